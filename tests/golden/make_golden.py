"""Writes tests/golden/codec_table.txt from the CPU oracle (and nothing else).

    python tests/golden/make_golden.py

The table freezes the oracle's byte codec: dequantized values of all 256 codes
and the codes of a grid of gradients, for S in {1, 8, 16}. Floats are written
in hexadecimal so they round-trip exactly.
"""
import os
import sys

HERE = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, os.path.dirname(os.path.dirname(HERE)))

import numpy as np  # noqa: E402

import oracle  # noqa: E402


def main():
    lines = ["# kind S arg value  (deq: code -> float hex; q: float hex -> code)",
             "# written by tests/golden/make_golden.py from the oracle's codec"]
    for S in (1.0, 8.0, 16.0):
        for q in range(-128, 128):
            lines.append(f"deq {S} {q} {float(oracle.dequantize(q, S)).hex()}")
        for g in np.concatenate([[0.0], np.logspace(-4, 8, 61), -np.logspace(-4, 8, 61)]):
            lines.append(f"q {S} {float(g).hex()} {oracle.quantize(float(g), S)}")
    with open(os.path.join(HERE, "codec_table.txt"), "w") as f:
        f.write("\n".join(lines) + "\n")


if __name__ == "__main__":
    main()
