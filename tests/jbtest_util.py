"""Helpers shared by the GPU tests: moving numpy arrays (fp32, or bf16 as uint16
bit patterns) to and from CUDA tensors, and the parity tolerances."""
from __future__ import annotations

import numpy as np

import oracle

# z: |z_gpu - z| <= 1e-6 absolute (fp32 Gaussians)
Z_ABS_TOL = 1e-6
# fp32 theta: |theta_gpu - theta| <= 2e-6 * (|theta_in| + sum_k |c_k z_k|); the scale is the
# size of the operands, which equals the size of the result when nothing cancels
F32_REL_TOL = 2e-6
# bf16 theta: at most one bf16 step apart
BF16_ULP_TOL = 1


def to_device(arr: np.ndarray):
    import torch
    if arr.dtype == np.float32:
        return torch.from_numpy(np.ascontiguousarray(arr)).cuda()
    if arr.dtype == np.uint16:
        return torch.from_numpy(np.ascontiguousarray(arr).view(np.int16)).cuda().view(torch.bfloat16)
    raise TypeError(arr.dtype)


def to_host(t) -> np.ndarray:
    import torch
    if t.dtype == torch.float32:
        return t.detach().cpu().numpy()
    if t.dtype == torch.bfloat16:
        return t.detach().view(torch.int16).cpu().numpy().view(np.uint16)
    raise TypeError(t.dtype)


def as_f64(arr: np.ndarray) -> np.ndarray:
    if arr.dtype == np.uint16:
        return oracle.bf16_to_f64(arr)
    return arr.astype(np.float64)


def bf16_ord(h: np.ndarray) -> np.ndarray:
    h = h.astype(np.int64)
    return np.where(h & 0x8000, -(h & 0x7FFF), h)


# Elements more than one bf16 step from the oracle that the fp32 allowance admits
# (reading R13: where theta + sum c z cancels, the bf16 steps of the result are finer
# than the fp32 error of the operands): (what, count, checked) per check_theta call.
WIDENED = []
# their largest share of the checked elements in any one call
BF16_WIDENED_SHARE = 1e-4


def check_theta(got: np.ndarray, want: np.ndarray, scale: np.ndarray, what: str = "",
                max_widened_share: float = BF16_WIDENED_SHARE) -> float:
    """Asserts parity; returns the worst error over its allowance (<= 1 passes)."""
    assert got.shape == want.shape and got.dtype == want.dtype
    if got.dtype == np.uint16:
        # one bf16 step of the result beyond the fp32 error allowance of the operands:
        # where theta + sum c z cancels, bf16 steps near the result are finer than the
        # fp32 error of z, and the allowance 2e-6 * scale decides
        d = np.abs(bf16_ord(got) - bf16_ord(want))
        w = as_f64(want)
        ulp = np.where(w == 0, 2.0**-133, np.ldexp(1.0, np.maximum(np.frexp(np.abs(w))[1] - 8, -133)))
        err = np.abs(as_f64(got) - w)
        r = np.where(d <= BF16_ULP_TOL, 0.0, err / (ulp + F32_REL_TOL * scale))
        worst = float(r.max()) if r.size else 0.0
        i = int(np.argmax(r)) if r.size else 0
        assert worst <= 1.0, f"{what}: bf16 distance {d[i]} at {i} (|d| {err[i]:.3e}, scale {scale[i]:.3e})"
        n_wide = int(np.count_nonzero(d > BF16_ULP_TOL))
        WIDENED.append((what, n_wide, int(d.size)))
        if n_wide:
            print(f"{what}: {n_wide} of {d.size} elements beyond one bf16 step, each within "
                  f"one step + 2e-6 x operands (share {n_wide / d.size:.2e})")
        assert n_wide <= max_widened_share * d.size + 1, \
            f"{what}: {n_wide} of {d.size} elements need the widened bf16 allowance"
        return max(worst, float(np.minimum(d, BF16_ULP_TOL).max(initial=0)) / BF16_ULP_TOL)
    d = np.abs(got.astype(np.float64) - want.astype(np.float64))
    allow = F32_REL_TOL * scale + 2.0**-149
    r = d / allow
    worst = float(r.max()) if r.size else 0.0
    i = int(np.argmax(r)) if r.size else 0
    assert worst <= 1.0, f"{what}: |d| {d[i]:.3e} > {allow[i]:.3e} at {i} (got {got[i]}, want {want[i]})"
    return worst


def update_scale(theta_in: np.ndarray, idx: np.ndarray, seeds, q, lr, denom, qscale) -> np.ndarray:
    """|theta_in| + sum_k |c_k z_k| at global indices idx (oracle Gaussians)."""
    s = as_f64(theta_in).__abs__()
    for sd, qq in zip(seeds, q):
        c = abs(oracle.coefficient(int(qq), lr, denom, qscale))
        s = s + c * np.abs(oracle.gaussian_at(sd, idx))
    return s
