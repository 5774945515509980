"""SPSA training loop of Algorithm 1 on the toy quadratic, on the CPU oracle.

Test infrastructure only. One replica stands for every machine: at the start
of an iteration each machine's copy equals the backup (Algorithm 1 copies
theta to theta_backup), so machine m evaluates its sample from the backup:
+eps, loss, -2 eps, loss, +eps; projected gradient (l+ - l-) / (2 eps);
one-byte code (Section 3). Then theta is restored from the backup and every
machine's (seed, byte) pair is applied in machine-timestamp order with weight
minus gradient times learning rate over the number of gradients (Algorithm 1).
Losses are summed in fp64.
"""
from __future__ import annotations

import dataclasses
from typing import List, Sequence

import numpy as np

import oracle


def quadratic_loss(theta: np.ndarray, a: np.ndarray, target: np.ndarray) -> float:
    d = theta.astype(np.float64) - target
    return float(0.5 * np.sum(a * d * d))


@dataclasses.dataclass
class StepRecord:
    seeds: List[tuple]
    ghat: List[float]
    codes: List[int]
    loss_after: float


def spsa_step(theta: np.ndarray, a, target, machine_ids: Sequence[int], step: int, eps: float,
              lr: float, qscale: float, denom: float | None = None) -> tuple[np.ndarray, StepRecord]:
    backup = theta.copy()
    seeds, ghat, codes = [], [], []
    for m in machine_ids:
        s = (int(m), step, 0)
        th = oracle.perturb(backup, 0, s, eps)
        lp = quadratic_loss(th, a, target)
        th = oracle.perturb(th, 0, s, -2 * eps)
        lm = quadratic_loss(th, a, target)
        g = (lp - lm) / (2 * eps)
        seeds.append(s)
        ghat.append(g)
        codes.append(oracle.quantize(g, qscale))
    K = len(seeds)
    out = oracle.update(backup, 0, seeds, np.array(codes, dtype=np.int8), lr,
                        float(K) if denom is None else denom, qscale)
    return out, StepRecord(seeds, ghat, codes, quadratic_loss(out, a, target))


def spsa_run(theta0: np.ndarray, a, target, machine_ids, n_steps: int, eps: float, lr: float,
             qscale: float) -> tuple[np.ndarray, List[StepRecord]]:
    theta = theta0.copy()
    recs = []
    for t in range(n_steps):
        theta, r = spsa_step(theta, a, target, machine_ids, t, eps, lr, qscale)
        recs.append(r)
    return theta, recs
