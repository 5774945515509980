"""Minimax polynomial coefficients for the Box-Muller transform in jb_rng.cuh.

    python paper_2306_10015_gb300/csrc/fit_poly.py

Method: the Remez exchange algorithm (E. Remez, 1934) for the weighted best
approximation by a linear combination of basis functions, in 40-digit
arithmetic (mpmath), then rounding each coefficient to fp32 and re-fitting
the remaining ones (a greedy correction for the rounding). Reported errors
are measured by evaluating the fp32 Horner schemes exactly as the kernel does
(each fused multiply-add rounded once to fp32) on a dense grid.

Fitted functions (the kernel's variables):
  R(w):  ln(1 + t) = -q (1 + w R(w)) / 4 ... written through q = -4 s,
         s = t / (2 + t), w = q^2, so that -2 ln(1 + t) = q + q w R(w);
         w in [0, 16 s_max^2], s in [-1/7, 1/5] (t in [-1/4, 1/2)).
  S(y):  sin(pi x / 4) = x (pi/4 + y S(y)), y = x^2, x in [0, 1]  (first octant);
         pi/4 is applied as hi + lo so that the leading term rounds once
  C(y):  cos(pi x / 4) = 1 + y C(y),  x in [0, 1], C of degree 3 (degree 8 in x;
         degree 2 saves one packed operation but leaves an absolute error of
         7.8e-8, too much of the 1e-6 budget of z at large radii once the radius
         comes from sqrt.approx)
"""
from __future__ import annotations

import struct

import mpmath as mp
import numpy as np

mp.mp.dps = 40


def f32(x) -> float:
    return float(np.float32(float(x)))


def remez(f, basis, a, b, weight, n_iter=25, grid=1200):
    """Coefficients c minimizing max |weight(x) (f(x) - sum c_i basis_i(x))| on [a, b]."""
    n = len(basis)
    # initial reference: Chebyshev extrema
    xs = [mp.mpf(a) + (mp.mpf(b) - a) * (1 - mp.cos(mp.pi * j / n)) / 2 for j in range(n + 1)]
    c = None
    for _ in range(n_iter):
        A = mp.matrix(n + 1, n + 1)
        rhs = mp.matrix(n + 1, 1)
        for j, x in enumerate(xs):
            for i, phi in enumerate(basis):
                A[j, i] = phi(x)
            A[j, n] = (-1) ** j / weight(x)
            rhs[j] = f(x)
        sol = mp.lu_solve(A, rhs)
        c = [sol[i] for i in range(n)]
        err = lambda x: weight(x) * (f(x) - sum(ci * phi(x) for ci, phi in zip(c, basis)))
        # locate the extrema of the error on a grid, one per sign run
        pts = [mp.mpf(a) + (mp.mpf(b) - a) * k / grid for k in range(grid + 1)]
        ev = [err(x) for x in pts]
        runs, cur = [], [0]
        for k in range(1, len(pts)):
            if mp.sign(ev[k]) == mp.sign(ev[cur[0]]) or ev[k] == 0:
                cur.append(k)
            else:
                runs.append(cur)
                cur = [k]
        runs.append(cur)
        ext = [max(r, key=lambda k: abs(ev[k])) for r in runs]
        while len(ext) > n + 1:  # drop the smallest extremum at an end
            if abs(ev[ext[0]]) < abs(ev[ext[-1]]):
                ext.pop(0)
            else:
                ext.pop()
        if len(ext) < n + 1:
            break
        new = [pts[k] for k in ext]
        if max(abs(u - v) for u, v in zip(new, xs)) < mp.mpf(b - a) / grid / 2:
            break
        xs = new
    return c


def fit_rounded(f, basis, a, b, weight):
    """Remez fit, then round coefficients to fp32 one at a time (lowest order first),
    re-fitting the rest around each rounded value."""
    fixed = []
    for i in range(len(basis)):
        rest = basis[i:]
        g = (lambda x, fixed=tuple(fixed): f(x) - sum(ci * phi(x) for ci, phi in zip(fixed, basis)))
        c = remez(g, rest, a, b, weight)
        fixed.append(mp.mpf(f32(c[0])))
    return [float(x) for x in fixed]


def fp32_fma(a, b, c):
    return np.float32(np.float64(a) * np.float64(b) + np.float64(c))


def hexf(x: float) -> str:
    return float(np.float32(x)).hex()


def main():
    # --- log: -2 ln(1 + t) = q + q w R(w), q = -4 t / (2 + t), w = q^2 -------------
    smax = mp.mpf(1) / 5
    wmax = 16 * smax ** 2
    # with s^2 = w / 16:  -2 ln(1+t) = -4 atanh(s) = q (1 + s^2/3 + s^4/5 + ...)
    #                     = q + q w R(w), R(w) = (atanh(s)/s - 1) / w
    def R_true(w):
        if w == 0:
            return mp.mpf(1) / 48
        s = mp.sqrt(w) / 4
        return (mp.atanh(s) / s - 1) / w
    basis = [lambda w, k=k: w ** k for k in range(3)]
    # weight: error of q w R relative to q, i.e. w * (R - P)
    Rc = fit_rounded(R_true, basis, 0, wmax, lambda w: w + mp.mpf("1e-30"))
    # --- sin(pi x / 4) = x S(x^2), x in [0, 1] ----------------------------------------
    def S_true(y):
        if y == 0:
            return mp.pi / 4
        x = mp.sqrt(y)
        return mp.sin(mp.pi * x / 4) / x
    # the leading coefficient is pi/4 itself, applied as a two-float pair (hi + lo)
    S_rest = lambda y: (S_true(y) - mp.pi / 4) / y if y != 0 else -(mp.pi / 4) ** 3 / 6
    Sr = fit_rounded(S_rest, [lambda y, k=k: y ** k for k in range(3)], 0, 1,
                     lambda y: (y + mp.mpf("1e-30")) / S_true(y))
    a_hi = f32(mp.pi / 4)
    a_lo = f32(mp.pi / 4 - mp.mpf(a_hi))
    Sc = [a_hi, a_lo] + Sr
    # --- cos(pi x / 4) = 1 + y C(y) ----------------------------------------------------
    def C_true(y):
        if y == 0:
            return -(mp.pi / 4) ** 2 / 2
        return (mp.cos(mp.pi * mp.sqrt(y) / 4) - 1) / y
    Cc = fit_rounded(C_true, [lambda y, k=k: y ** k for k in range(4)], 0, 1,
                     lambda y: (y + mp.mpf("1e-30")) / mp.cos(mp.pi * mp.sqrt(y) / 4))

    # --- measured fp32 errors of the Horner schemes ------------------------------------
    x = np.linspace(0, 1, 200001, dtype=np.float64).astype(np.float32)
    y = (x.astype(np.float64) ** 2).astype(np.float32)
    def horner(cs, v):
        p = np.full_like(v, np.float32(cs[-1]))
        for c in cs[-2::-1]:
            p = fp32_fma(v, p, np.float32(c))
        return p
    # S = fma(x, a_hi, x * (a_lo + y (s1 + y (s2 + y s3))))
    inner = horner([Sc[1]] + Sc[2:], y)
    S = fp32_fma(x, np.float32(Sc[0]), (x.astype(np.float64) * inner.astype(np.float64)).astype(np.float32))
    C = fp32_fma(y, horner(Cc, y), np.float32(1.0))
    xs = x.astype(np.float64)
    es = np.max(np.abs(S[1:] - np.sin(np.pi * xs[1:] / 4)) / np.sin(np.pi * xs[1:] / 4))
    ec = np.max(np.abs(C - np.cos(np.pi * xs / 4)) / np.cos(np.pi * xs / 4))
    t = np.linspace(-0.25, 0.5, 300001)[:-1].astype(np.float32)
    q = (-4 * t.astype(np.float64) / (2 + t.astype(np.float64))).astype(np.float32)
    w = (q.astype(np.float64) ** 2).astype(np.float32)
    Lp = fp32_fma(q, (w.astype(np.float64) * horner(Rc, w)).astype(np.float32), q)  # degree 2
    ref = -2 * np.log1p(t.astype(np.float64))
    nz = ref != 0
    el = np.max(np.abs(Lp[nz] - ref[nz]) / np.abs(ref[nz]))
    print("// R (log):", ", ".join(hexf(c) for c in Rc), f"   max rel err {el:.3e} (q exact)")
    print("// S (sin):", ", ".join(hexf(c) for c in Sc), f"   max rel err {es:.3e}")
    print("// C (cos):", ", ".join(hexf(c) for c in Cc), f"   max rel err {ec:.3e}")
    for name, cs in (("kLogR", Rc), ("kSinS", Sc), ("kCosC", Cc)):
        print(f"constexpr float {name}[{len(cs)}] = {{" + ", ".join(hexf(c) + "f" for c in cs) + "};")


if __name__ == "__main__":
    main()
