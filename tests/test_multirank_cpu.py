"""The N > 1 path on the CPU with gloo, world size 2.

* bench.py's whole-job aggregation over replica ranks: slowest time, summed units.
* The method's data-parallel exchange (Section 2; Algorithm 1): each rank is a
  machine; it evaluates its own SPSA sample on the toy quadratic with the
  oracle, quantizes it to one byte, the (seed, byte) pairs are all-gathered
  (standing in for the method's exchange step), and every rank applies the full
  list. The replicas must stay bitwise identical (checksum and bytes).
"""
import os
import socket

import numpy as np
import pytest
import torch
import torch.distributed as dist
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _init(rank, world, port):
    import sys
    sys.path.insert(0, ROOT)
    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    dist.init_process_group("gloo", rank=rank, world_size=world)


def _aggregate_worker(rank, world, port, q):
    _init(rank, world, port)
    import bench
    ms, units = bench.aggregate_ranks(10.0 + 5.0 * rank, 100.0 * (rank + 1), dist, torch.device("cpu"))
    q.put((rank, ms, units))
    dist.destroy_process_group()


def _replica_worker(rank, world, port, q):
    _init(rank, world, port)
    import oracle
    from oracle import spsa
    import synthetic
    toy = synthetic.toy_quadratic(1 << 12)
    mids = synthetic.toy_machine_ids()[:world]
    theta = toy.theta0.copy()
    eps, lr, qs = 1e-3, 1e-3, 16.0
    for t in range(3):
        backup = theta.copy()
        s = (int(mids[rank]), t, 0)  # this rank is machine `rank`
        th = oracle.perturb(backup, 0, s, eps)
        lp = spsa.quadratic_loss(th, toy.a, toy.target)
        th = oracle.perturb(th, 0, s, -2 * eps)
        lm = spsa.quadratic_loss(th, toy.a, toy.target)
        code = oracle.quantize((lp - lm) / (2 * eps), qs)
        pairs = [None] * world
        dist.all_gather_object(pairs, (s, code))  # 17 bytes of payload per machine
        seeds = [p[0] for p in pairs]
        codes = np.array([p[1] for p in pairs], dtype=np.int8)
        theta = oracle.update(backup, 0, seeds, codes, lr, float(world), qs)
    h = oracle.checksum([theta], [0])
    all_h = [None] * world
    dist.all_gather_object(all_h, (h, theta.tobytes()))
    q.put((rank, all_h))
    dist.destroy_process_group()


def _run(fn, world=2):
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = free_port()
    procs = [ctx.Process(target=fn, args=(r, world, port, q)) for r in range(world)]
    for p in procs:
        p.start()
    out = [q.get(timeout=240) for _ in procs]
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    return sorted(out, key=lambda x: x[0])


def test_whole_job_aggregation_gloo():
    out = _run(_aggregate_worker)
    for _, ms, units in out:
        assert ms == 15.0 and units == 300.0


def test_replicas_stay_identical_gloo():
    out = _run(_replica_worker)
    (_, hs0), (_, hs1) = out
    assert hs0 == hs1
    (h0, b0), (h1, b1) = hs0
    assert h0 == h1 and b0 == b1
