"""Prints the fp32 level and midpoint table of the 4-bit weight code (jb_q4.cu).

    python paper_2306_10015_gb300/csrc/gen_q4_levels.py

Levels: quantiles of N(0,1) (scipy.special.ndtri) at probabilities
delta + (1/2 - delta) j / 7 (j = 0..7, the last is the median, exactly 0) and
1/2 + (1/2 - delta) j / 8 (j = 1..8), divided by the largest so they span
[-1, 1], delta = 1/32, rounded to fp32. Midpoints: (L_j + L_{j+1}) / 2 of the
fp32 levels, computed in double and rounded to fp32.
"""
import numpy as np
from scipy.special import ndtri


def levels() -> np.ndarray:
    d = 1.0 / 32.0
    neg = ndtri(d + (0.5 - d) * np.arange(8) / 7.0)
    pos = ndtri(0.5 + (0.5 - d) * np.arange(1, 9) / 8.0)
    v = np.concatenate([neg, pos])
    v[7] = 0.0
    out = (v / v[-1]).astype(np.float32)
    out[7], out[15] = 0.0, 1.0
    return out


def main():
    lev = levels()
    mid = ((lev[:-1].astype(np.float64) + lev[1:].astype(np.float64)) / 2).astype(np.float32)
    print("constexpr float kQ4Level[16] = {" + ", ".join(float(x).hex() + "f" for x in lev) + "};")
    print("constexpr float kQ4Mid[15] = {" + ", ".join(float(x).hex() + "f" for x in mid) + "};")


if __name__ == "__main__":
    main()
