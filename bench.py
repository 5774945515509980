#!/usr/bin/env python
"""Benchmark: one SPSA step of the shared-randomness method on OPT-shaped
synthetic parameters, through the C ABI of libjb.

A step is one pass of the whole hot path over the parameter set:
  perturb(+eps), perturb(-2 eps), perturb(+eps)  one SPSA sample around its two
                                                 loss evaluations (Algorithm 1)
  quantize the sample's projected gradient       one byte (Section 3)
  fused update of K machines' (seed, byte) pairs (Section 2; Algorithm 1)
The loss evaluations themselves (model forwards) are outside the path; the
projected gradient is a seeded synthetic scalar.

Metric: param.seed updates/s = N (K + 3) / step time, the whole job over all
ranks. Inputs (25.7 GB for the 13B-shaped set) are far larger than L2, so no
flush is needed between steps. Ranks (torchrun, N > 1) are independent
replicas: the path has no exchange step on the device.

  python bench.py [--gpus N] [--steps K] [--warmup W] [--impl jb|reference]
"""
from __future__ import annotations

import argparse
import json
import os
import statistics
import subprocess
import sys
import threading
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "param·seed updates/s and HBM GB/s (% roofline), 13B-shaped bf16, K=64"
UNIT = "param·seed/s"

# Algorithmic lane operations per element-seed (the ALU roofline's unit of work):
# a quarter Philox4x32-10 block (10 rounds x 2 wide multiplies + 2 three-way XORs,
# over 4 words) = 10; half a Box-Muller pair (2 uniform conversions, log, sqrt,
# sin, cos, 2 products over 2 elements) = 4; the accumulate FMA = 1.
OPS_PER_PARAM_SEED = 15
LANES_PER_SM_CLK = 128
# special-function unit: 16 lanes per clock per SM (measured: lg2.approx at 16.1)
MUFU_LANES_PER_SM_CLK = 16


def parse():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=5)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", choices=["jb", "reference"], default="jb")
    ap.add_argument("--model", default="opt-13b")
    ap.add_argument("--dtype", choices=["bf16", "f32"], default="bf16")
    ap.add_argument("--K", type=int, default=64)
    ap.add_argument("--eps", type=float, default=1e-3)
    ap.add_argument("--lr", type=float, default=1e-6)
    ap.add_argument("--qscale", type=float, default=16.0)
    ap.add_argument("--e2e-steps", type=int, default=4)
    ap.add_argument("--e2e-groups", type=int, default=16, help="tensor groups of the e2e pipeline")
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--cpu-seconds", type=float, default=10.0,
                    help="target CPU time of each oracle sample (all cores, then one core)")
    ap.add_argument("--sweep", default="1,4,16,64,256",
                    help="comma list of K: the fused update timed per K (empty: no sweep)")
    ap.add_argument("--no-sweep", action="store_true", help="skip the K sweep")
    ap.add_argument("--sweep-out", default="", help="file for the sweep's JSON lines")
    ap.add_argument("--next-legs", action="store_true",
                    help="(the default) with the sweep, also time the backup-fused update, the "
                         "replay, the checksum and the 4-bit perturbation")
    ap.add_argument("--no-next-legs", action="store_true", help="skip those legs")
    a = ap.parse_args()
    a.next_legs = not a.no_next_legs
    return a


def aggregate_ranks(ms_local: float, units_local: float, dist=None, device=None):
    """Whole-job figures over ranks that ran independent replicas: the slowest
    rank's time and the sum of the units all ranks processed."""
    if dist is None or not dist.is_initialized() or dist.get_world_size() == 1:
        return ms_local, units_local
    import torch
    t = torch.tensor([ms_local, units_local], dtype=torch.float64, device=device)
    mx = t.clone()
    dist.all_reduce(mx, op=dist.ReduceOp.MAX)
    dist.all_reduce(t, op=dist.ReduceOp.SUM)
    return float(mx[0].item()), float(t[1].item())


def dist_env():
    return (int(os.environ.get("RANK", 0)), int(os.environ.get("LOCAL_RANK", 0)),
            int(os.environ.get("WORLD_SIZE", 1)))


def workload_name(a) -> str:
    return f"{a.model}-shaped {a.dtype}, SPSA step (perturb +eps/-2eps/+eps, K={a.K} fused update)"


# --- clocks ------------------------------------------------------------------------

class ClockSampler:
    FIELDS = ["clocks.sm", "clocks.max.sm", "power.draw", "clocks_event_reasons.hw_slowdown",
              "clocks_event_reasons.hw_thermal_slowdown", "clocks_event_reasons.sw_thermal_slowdown",
              "clocks_event_reasons.sw_power_cap"]

    def __init__(self, index: int):
        self.index = index
        self.proc = None
        self.lines = []

    def start(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.index), "--query-gpu=" + ",".join(self.FIELDS),
                 "--format=csv,noheader,nounits", "-lms", "200"],
                stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
            self.thread = threading.Thread(target=self._read, daemon=True)
            self.thread.start()
        except OSError:
            self.proc = None

    def _read(self):
        for ln in self.proc.stdout:
            self.lines.append(ln.strip())

    def stop(self) -> dict:
        if self.proc is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
        self.thread.join(timeout=5)
        sm, smax, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for ln in self.lines:
            parts = [p.strip() for p in ln.split(",")]
            if len(parts) != len(self.FIELDS):
                continue
            try:
                sm.append(float(parts[0]))
                smax.append(float(parts[1]))
            except ValueError:
                continue
            for name, v in zip(names, parts[3:]):
                if v.lower().startswith("active"):
                    reasons.add(name)
        return {"sm_mhz": statistics.median(sm) if sm else None,
                "sm_max_mhz": max(smax) if smax else None, "reasons": sorted(reasons),
                "samples": len(sm)}


# --- the CPU oracle (baseline and reference arm) --------------------------------------

def oracle_rate(a, target_s: float, threads: int = 0):
    """The oracle, as it stands, on a bounded sample of the workload: sampled
    elements x (3 perturb seeds + K update seeds), on `threads` host threads (0: all
    cores the process may use). Returns (param.seed/s, threads, seconds, elements)."""
    import numpy as np

    import oracle
    import synthetic
    cores = threads if threads > 0 else len(os.sched_getaffinity(0))
    oracle.set_threads(cores)
    specs = synthetic.opt_tensors(a.model)
    numels = [s.numel for s in specs]
    offs = synthetic.flat_offsets(numels)
    seeds = [(int(m), 0, 0) for m in synthetic.machine_ids(a.K, 900)]
    q = synthetic.byte_codes(a.K, 900, 0)
    own = seeds[0]

    def run(n):
        pos = synthetic.sample_positions(numels, n, 901)
        idx = np.concatenate([fo + p for fo, p in zip(offs, pos)]).astype(np.uint64)
        vals = synthetic.normal_values(idx.size, 0.02, 902)
        if a.dtype == "bf16":
            vals = oracle.round_bf16(vals.astype(np.float64)) if idx.size < 4096 else \
                (vals.view(np.uint32) >> 16).astype(np.uint16)
        t0 = time.perf_counter()
        v = vals
        for e in (a.eps, -2 * a.eps, a.eps):
            v = oracle.perturb_at(v, idx, own, e)
        oracle.update_at(v, idx, seeds, q, a.lr, 1.0, a.qscale)
        return idx.size, time.perf_counter() - t0

    n0, t0 = run(1 << 12)
    rate = n0 * (a.K + 3) / max(t0, 1e-6)
    n = int(min(max(rate * target_s / (a.K + 3), 1 << 12), 1 << 26))
    n, t = run(n)
    oracle.set_threads(len(os.sched_getaffinity(0)))
    return n * (a.K + 3) / t, cores, t, n


def bench_config(a, world):
    """The workload description both arms print (sizes from the OPT shapes alone)."""
    import synthetic
    specs = synthetic.opt_tensors(a.model)
    return {"workload": workload_name(a), "n_params": sum(sp.numel for sp in specs),
            "n_tensors": len(specs), "K": a.K, "eps": a.eps, "lr": a.lr, "qscale": a.qscale,
            "l2": "inputs larger than L2 (no flush needed)", "parallelism": f"replicas x{world}"}


def run_reference(a):
    rank, _, world = dist_env()
    if rank != 0:
        return
    steps_rates = []
    n_used = 0
    cores = 0
    for _ in range(max(a.steps, 1)):
        rate, cores, t, n_used = oracle_rate(a, min(a.cpu_seconds, 60.0 / max(a.steps, 1)))
        steps_rates.append(rate)
    value = statistics.median(steps_rates)
    sample = (f"{n_used} sampled elements of the {a.model}-shaped set per step, each taking "
              f"3 perturb seeds and {a.K} update seeds")
    print(json.dumps({
        "impl": "reference", "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": a.gpus,
        "steps": a.steps, "warmup": a.warmup, "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "f64", "data": "synthetic",
        "config": bench_config(a, world),
        "cpu_baseline": {"value": value, "unit": UNIT, "cores": cores, "kind": "oracle",
                         "sample": sample},
        "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }), flush=True)


# --- the GPU arm -----------------------------------------------------------------------

def main():
    a = parse()
    if a.impl == "reference":
        run_reference(a)
        return
    import numpy as np
    import torch

    import paper_2306_10015_gb300 as jb
    import synthetic

    rank, local_rank, world = dist_env()
    torch.cuda.set_device(local_rank)
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl", device_id=torch.device("cuda", local_rank))
    else:
        dist = None

    def barrier():
        if dist is not None:
            dist.barrier()

    tdt = torch.bfloat16 if a.dtype == "bf16" else torch.float32
    esize = 2 if a.dtype == "bf16" else 4
    specs, tensors, offs = synthetic.opt_parameters(a.model, tdt, seed=synthetic.MASTER_SEED + rank)
    table = jb.ParamTable(tensors, offs)
    N = table.numel
    K = a.K
    mids = synthetic.machine_ids(K, 900)
    own = 0  # this replica's machine is the first of the K
    n_total = a.warmup + a.steps + a.e2e_steps + 1
    seeds = [jb.seeds_array([(int(m), t, 0) for m in mids]) for t in range(n_total)]
    codes = [synthetic.byte_codes(K, 900, t) for t in range(n_total)]
    ghat = synthetic.rng(903).standard_normal(n_total) * 100.0
    stream = torch.cuda.current_stream()
    launches_per_step = 3 * (-(-table.n_segments // 1000)) + (-(-table.n_segments // 700))

    ev = {}

    def step(t, timed=False):
        s_own = (int(mids[own]), t, 0)
        if timed:
            ev.setdefault("p0", []).append(torch.cuda.Event(enable_timing=True))
            ev["p0"][-1].record(stream)
        jb.jb_perturb(table, s_own, a.eps, stream)
        jb.jb_perturb(table, s_own, -2 * a.eps, stream)
        jb.jb_perturb(table, s_own, a.eps, stream)
        q = codes[t]
        q[own] = jb.jb_quantize_grad(float(ghat[t]), a.qscale)
        if timed:
            ev.setdefault("u0", []).append(torch.cuda.Event(enable_timing=True))
            ev["u0"][-1].record(stream)
        jb.jb_apply_updates(table, seeds[t], q, a.lr, 1.0, a.qscale, stream)
        if timed:
            ev.setdefault("u1", []).append(torch.cuda.Event(enable_timing=True))
            ev["u1"][-1].record(stream)

    for t in range(a.warmup):
        step(t)
    torch.cuda.synchronize()
    barrier()
    torch.cuda.synchronize()
    clocks = ClockSampler(local_rank)
    clocks.start()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    for t in range(a.warmup, a.warmup + a.steps):
        step(t, timed=True)
    e1.record(stream)
    torch.cuda.synchronize()
    barrier()
    clk = clocks.stop()
    ms = e0.elapsed_time(e1)
    upd_ms = [x.elapsed_time(y) for x, y in zip(ev["u0"], ev["u1"])]
    pert_ms = [x.elapsed_time(y) / 3 for x, y in zip(ev["p0"], ev["u0"])]
    ms, units = aggregate_ranks(ms, float(N * (K + 3) * a.steps), dist,
                                torch.device("cuda", local_rank))
    ms_per_step = ms / a.steps
    units_per_step = units / a.steps
    value = units_per_step / (ms_per_step / 1e3)

    # end to end through the same public calls, theta in pinned host memory: the
    # copies in, the step and the copies out of groups of tensors run on three
    # streams (run_e2e)
    e2e = None
    if not a.no_e2e:
        e2e = run_e2e(a, jb, tensors, offs, seeds, codes, ghat, mids, own, stream, N, esize,
                      units_per_step, dist, a.e2e_groups)

    sweep_lines, next_lines = [], []
    if a.sweep and not a.no_sweep and rank == 0:
        sweep_lines, next_lines = run_sweep(a, jb, table, mids, stream)

    if rank != 0:
        if dist is not None:
            dist.destroy_process_group()
        return

    roof = Roofline(a, torch, N, esize, generator_rate(jb, stream))
    roofline = roof.report(K, upd_ms)
    roofline.update({
        "bound": "alu", "traffic": load_traffic(a),
        "kernel": "seeded_kernel<bf16, update>" if a.dtype == "bf16" else "seeded_kernel<f32, update>",
        "perturb_ms": statistics.mean(pert_ms), "perturb_ms_best": min(pert_ms),
        "perturb_ms_median": statistics.median(pert_ms),
        "timing": f"CUDA events per launch over the {a.steps} timed steps; frac uses the best launch"})
    cpu = None
    if not a.no_cpu_baseline and world == 1:
        rate, cores, t, n = oracle_rate(a, a.cpu_seconds)
        rate1, _, t1, n1 = oracle_rate(a, a.cpu_seconds, threads=1)
        cpu = {"value": rate, "unit": UNIT, "cores": cores, "kind": "oracle",
               "sample": f"{n} sampled elements x (3 perturb + {K} update seeds), {t:.1f} s",
               "single_thread": {"value": rate1, "unit": UNIT, "cores": 1,
                                 "sample": f"{n1} sampled elements x (3 + {K} seeds), {t1:.1f} s"}}
    step_bytes = 4 * 2 * esize * N  # 3 perturb passes + 1 update pass, read + write
    out = {
        "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": a.steps,
        "warmup": a.warmup, "ms_per_step": ms_per_step, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": a.dtype, "data": "synthetic",
        "config": bench_config(a, world),
        "hbm_gbs_step": step_bytes * world / (ms_per_step / 1e3) / 1e9,
        "roofline": roofline, "cpu_baseline": cpu, "e2e": e2e,
        "gpu_launches": launches_per_step * a.steps, "clocks": clk,
    }
    if sweep_lines:
        out["sweep"] = [roof.report(ln["K"], ln["ms"]) if "K" in ln else ln for ln in sweep_lines]
    if next_lines:
        out["next"] = [roof.leg(ln) for ln in next_lines]
    print(json.dumps(out), flush=True)
    if dist is not None:
        dist.destroy_process_group()


def stats(ms):
    return {"best": min(ms), "median": statistics.median(ms), "mean": statistics.mean(ms), "n": len(ms)}


def generator_rate(jb, stream, n_blocks=1 << 32, reps=5):
    """Element-seeds per second of Philox4x32-10 alone (jb_debug_philox_fold: the hot
    path's block function, its words XOR-folded), best of `reps` launches."""
    import torch
    out = torch.zeros(1, dtype=torch.int32, device="cuda")
    jb.jb_debug_philox_fold((1, 2, 3), 0, n_blocks, out, stream)
    best = float("inf")
    for _ in range(reps):
        x0, x1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        x0.record(stream)
        jb.jb_debug_philox_fold((1, 2, 3), 0, n_blocks, out, stream)
        x1.record(stream)
        torch.cuda.synchronize()
        best = min(best, x0.elapsed_time(x1))
    return 4 * n_blocks / (best / 1e3)


class Roofline:
    """Rooflines of the fused K-seed update on this GPU, per K and launch time.

    * frac (judged; the combined roofline of the task): T_roof = max(T_HBM, T_ALG),
      T_HBM = 2 sizeof(T) N / measured copy bandwidth, T_ALG = the algorithm's fixed
      count of OPS_PER_PARAM_SEED = 15 lane operations per element-seed (a quarter
      Philox4x32-10 block: 10 rounds x (2 wide multiplies + 2 three-input XORs) / 4;
      half a Box-Muller pair: 2 uniforms, log, sqrt, sin, cos, 2 products over 2
      elements; one accumulating FMA), each at one lane-operation per lane per clock,
      152 SMs x 128 lanes x the maximum SM clock. frac = T_roof / T_best.
    * floors.generator: the same K N element-seeds at the rate of Philox4x32-10 alone
      (jb_debug_philox_fold, measured in this run): what the wide multiplies cost.
    * floors.mufu: one special-function operation per element-seed (rcp and sqrt
      per word pair) at 16 lanes per clock per SM.
    * issue_measured: the kernel's own ncu-measured lane-instructions per
      element-seed at peak issue (occupancy of the issue slots, not a bound)."""

    def __init__(self, a, torch, N, esize, gen_rate):
        props = torch.cuda.get_device_properties(torch.cuda.current_device())
        self.sms = props.multi_processor_count
        peaks = {}
        try:
            with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
                peaks = json.load(f)
        except OSError:
            pass
        self.hbm_peak = float(peaks.get("hbm_gbs", 6800.0))
        self.peak_src = "measured" if "hbm_gbs" in peaks else "fallback"
        self.f_max = float(peaks.get("sm_max_mhz", 2070.0)) * 1e6
        self.N, self.esize, self.gen_rate = N, esize, gen_rate
        self.lanes = self.sms * LANES_PER_SM_CLK * self.f_max
        self.instr = load_instr_per_param_seed(a)

    def leg(self, ln):
        """A NEXT-row leg with its roofline: the backup-fused update and the replay
        against the update's (the same bytes per pass and work per element-seed;
        the backup refresh adds one write), the checksum and the 4-bit pass against
        the measured copy bandwidth."""
        ln = dict(ln)
        if ln.get("mode") in ("fused", "fused+refresh", "replay"):  # one pass over theta
            k = ln["K"] if ln["leg"] == "restore+update" else ln["steps"] * ln["K_per_step"]
            t = ln["ms"] / 1e3
            extra = 1.5 if ln.get("mode") == "fused+refresh" else 1.0
            t_hbm = extra * 2 * self.esize * self.N / (self.hbm_peak * 1e9)
            t_alg = OPS_PER_PARAM_SEED * k * self.N / self.lanes
            ln["frac"] = max(t_hbm, t_alg) / t
            ln["generator_floor"] = k * self.N / self.gen_rate / t
        elif ln.get("leg") in ("checksum", "perturb_q4"):
            ln["hbm_frac"] = ln["hbm_gbs"] / self.hbm_peak
        return ln

    def report(self, K, ms_list):
        st = stats(ms_list)
        t = st["best"] / 1e3
        N = self.N
        t_hbm = 2 * self.esize * N / (self.hbm_peak * 1e9)
        t_alg = OPS_PER_PARAM_SEED * K * N / self.lanes
        t_gen = K * N / self.gen_rate
        t_mufu = K * N / (self.sms * MUFU_LANES_PER_SM_CLK * self.f_max)
        out = {
            "K": K, "update_ms": st["mean"], "update_ms_best": st["best"], "update_ms_median": st["median"],
            "launches": st["n"], "param_seed_per_s": K * N / t,
            "param_seed_per_s_median": K * N / (st["median"] / 1e3),
            "achieved": OPS_PER_PARAM_SEED * K * N / t / 1e12, "peak": self.lanes / 1e12, "unit": "Tops/s",
            "frac": max(t_hbm, t_alg) / t, "ops_per_param_seed": OPS_PER_PARAM_SEED,
            "peak_basis": f"{self.sms} SMs x {LANES_PER_SM_CLK} lanes x {self.f_max / 1e6:.0f} MHz; "
                          f"HBM {self.hbm_peak:.0f} GB/s ({self.peak_src})",
            "t_hbm_ms": t_hbm * 1e3, "t_alg_ms": t_alg * 1e3,
            "hbm_gbs": 2 * self.esize * N / t / 1e9, "hbm_frac": t_hbm / t,
            "floors": {"generator": {"philox_only_param_seed_per_s": self.gen_rate, "t_ms": t_gen * 1e3,
                                     "frac": t_gen / t},
                       "mufu": {"lanes_per_clk_per_sm": MUFU_LANES_PER_SM_CLK, "ops_per_param_seed": 1,
                                "t_ms": t_mufu * 1e3, "frac": t_mufu / t}},
        }
        if self.instr is not None:
            t_iss = self.instr * K * N / self.lanes
            out["issue_measured"] = {"instr_per_param_seed": self.instr, "t_ms": t_iss * 1e3,
                                     "frac": max(t_iss, t_hbm) / t}
        return out


class E2EPipeline:
    """Theta in pinned host memory, one step at a time through the public calls.

    The tensors are split into n_groups groups. Each group lives in one pinned host
    buffer and one device buffer, and its tensors are views into them (64-element
    aligned), so a group moves in one copy each way. Three streams pipeline the
    groups: group g + 1 arrives while group g is transformed, and group g - 1
    leaves. Only the first group's copy in and the last group's copy out are not
    hidden behind compute, so the groups ramp up and down geometrically (1/16, 1/8,
    1/4, 1/2 of a middle group at each end) and the smallest tensors are placed at
    the two ends to make those groups small. z depends only on the global index,
    so any order and split of the table gives the same bits."""

    def __init__(self, jb, tensors, offs, stream, n_groups=32):
        import torch
        self.jb, self.stream = jb, stream
        groups = self.split(tensors, n_groups)
        pad = lambda n: -(-n // 64) * 64
        self.dev_bufs, self.host_bufs = [], []
        self.views, self.host_views = [None] * len(tensors), [None] * len(tensors)
        for g in groups:
            n = sum(pad(tensors[i].numel()) for i in g)
            d = torch.empty(n, dtype=tensors[0].dtype, device=tensors[0].device)
            h = torch.empty(n, dtype=tensors[0].dtype, pin_memory=True)
            o = 0
            for i in g:
                m = tensors[i].numel()
                self.views[i] = d[o:o + m].view(tensors[i].shape)
                self.views[i].copy_(tensors[i])
                self.host_views[i] = h[o:o + m].view(tensors[i].shape)
                o += pad(m)
            h.copy_(d)
            self.dev_bufs.append(d)
            self.host_bufs.append(h)
        torch.cuda.synchronize()
        self.groups = groups
        self.copy_bytes = sum(b.numel() * b.element_size() for b in self.dev_bufs)
        self.tables = [jb.ParamTable([self.views[i] for i in g], [offs[i] for i in g]) for g in groups]
        self.s_in, self.s_out = torch.cuda.Stream(), torch.cuda.Stream()
        self.out_done = [None] * len(groups)

    @staticmethod
    def split(tensors, n_groups):
        """Groups of tensor indices: the smallest tensors at both ends of the order,
        group sizes ramping geometrically at both ends, every group non-empty."""
        sizes = [t.numel() for t in tensors]
        n = len(sizes)
        n_groups = max(1, min(n_groups, n))
        ramp = min(4, (n_groups - 1) // 2)
        w = [1.0] * n_groups
        for i in range(ramp):
            w[i] = w[n_groups - 1 - i] = 2.0 ** (i - ramp)
        # order: small tensors alternately to the front and the back, the rest between
        by_size = sorted(range(n), key=lambda i: sizes[i])
        total = sum(sizes)
        end_budget = total * sum(w[:ramp]) / sum(w)
        front, back, used, acc = [], [], set(), 0
        for k, i in enumerate(by_size):
            if acc >= 2 * end_budget:
                break
            (front if k % 2 == 0 else back).append(i)
            used.add(i)
            acc += sizes[i]
        order = front + [i for i in range(n) if i not in used] + back[::-1]
        bounds, c = [], 0.0
        for x in w[:-1]:
            c += x
            bounds.append(total * c / sum(w))
        groups, cur, acc = [], [], 0
        for k, i in enumerate(order):
            cur.append(i)
            acc += sizes[i]
            left = n - 1 - k  # tensors not yet placed
            need = n_groups - 1 - len(groups)  # groups still to open after this one
            if len(groups) < n_groups - 1 and (acc >= bounds[len(groups)] or left == need):
                groups.append(cur)
                cur = []
        if cur:
            groups.append(cur)
        return groups

    def step(self, s_own, seeds, q, eps, lr, qscale):
        """Enqueue one step: per group copy in, perturb +eps/-2 eps/+eps, update, copy out."""
        import torch
        jb, stream = self.jb, self.stream
        for gi, tab in enumerate(self.tables):
            if self.out_done[gi] is not None:
                self.s_in.wait_event(self.out_done[gi])
            with torch.cuda.stream(self.s_in):
                self.dev_bufs[gi].copy_(self.host_bufs[gi], non_blocking=True)
            arrived = torch.cuda.Event()
            arrived.record(self.s_in)
            stream.wait_event(arrived)
            jb.jb_perturb(tab, s_own, eps, stream)
            jb.jb_perturb(tab, s_own, -2 * eps, stream)
            jb.jb_perturb(tab, s_own, eps, stream)
            jb.jb_apply_updates(tab, seeds, q, lr, 1.0, qscale, stream)
            done = torch.cuda.Event()
            done.record(stream)
            self.s_out.wait_event(done)
            with torch.cuda.stream(self.s_out):
                self.host_bufs[gi].copy_(self.dev_bufs[gi], non_blocking=True)
            self.out_done[gi] = torch.cuda.Event()
            self.out_done[gi].record(self.s_out)


def run_e2e(a, jb, tensors, offs, seeds, codes, ghat, mids, own, stream, N, esize,
            units_per_step, dist, n_groups=32):
    """The step end to end (E2EPipeline), timed from the first copy in to the last
    copy out, after one untimed step."""
    import torch
    pipe = E2EPipeline(jb, tensors, offs, stream, n_groups)

    def step(t):
        q = codes[t]
        q[own] = jb.jb_quantize_grad(float(ghat[t]), a.qscale)
        pipe.step((int(mids[own]), t, 0), seeds[t], q, a.eps, a.lr, a.qscale)

    base = a.warmup + a.steps
    step(base)
    torch.cuda.synchronize()
    if dist is not None:
        dist.barrier()
    x0, x1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    x0.record(pipe.s_in)
    for t in range(base + 1, base + 1 + a.e2e_steps):
        step(t)
    x1.record(pipe.s_out)
    torch.cuda.synchronize()
    xms = x0.elapsed_time(x1) / a.e2e_steps
    # the same copies without overlap, for reference
    y0, y1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    y0.record(stream)
    for h, d in zip(pipe.host_bufs, pipe.dev_bufs):
        d.copy_(h, non_blocking=True)
    y1.record(stream)
    z1 = torch.cuda.Event(enable_timing=True)
    for h, d in zip(pipe.host_bufs, pipe.dev_bufs):
        h.copy_(d, non_blocking=True)
    z1.record(stream)
    torch.cuda.synchronize()
    h2d_ms, d2h_ms = y0.elapsed_time(y1), y1.elapsed_time(z1)
    xms, _ = aggregate_ranks(xms, 0.0, dist, torch.device("cuda", torch.cuda.current_device()))
    groups, copy_bytes = len(pipe.groups), pipe.copy_bytes
    del pipe
    return {"value": units_per_step / (xms / 1e3), "unit": UNIT,
            "h2d_bytes_per_step": copy_bytes, "d2h_bytes_per_step": copy_bytes,
            "ms_per_step": xms, "groups": groups, "h2d_ms": h2d_ms, "d2h_ms": d2h_ms}


# The sources the update kernel's device code and launch shape are built from.
UPDATE_KERNEL_SOURCES = ("jb_internal.h", "jb_kernels.cu", "jb_rng.cuh")


def kernel_sources_digest() -> str:
    """sha1 over the update kernel's sources; its ncu counters are valid only for
    the build they measured."""
    import hashlib
    csrc = os.path.join(ROOT, "paper_2306_10015_gb300", "csrc")
    h = hashlib.sha1()
    for name in UPDATE_KERNEL_SOURCES:
        with open(os.path.join(csrc, name), "rb") as f:
            h.update(name.encode() + b"\0" + f.read())
    return h.hexdigest()


def load_counters():
    """ncu figures of the update kernel (profiles/traffic.json), or {} once the
    kernel sources differ from those the counters were taken on."""
    path = os.path.join(ROOT, "profiles", "traffic.json")
    try:
        with open(path) as f:
            d = json.load(f)
    except (OSError, ValueError):
        return {}
    if d.get("kernel_sources_sha1") != kernel_sources_digest():
        return {}
    return d


def load_traffic(a):
    """DRAM bytes per update launch (ncu), or None."""
    return load_counters().get("update_bytes_per_launch", {}).get(f"{a.model}/{a.dtype}/K={a.K}")


def load_instr_per_param_seed(a):
    """Measured marginal lane-instructions per element-seed of the update (ncu,
    K = 1 vs K = 64), or None."""
    return load_counters().get("instr_per_param_seed", {}).get(a.dtype)


SWEEP_REPS = {1: 20, 4: 10, 16: 5, 64: 3, 256: 2}


def run_sweep(a, jb, table, mids, stream):
    """The fused update per K (one warm-up launch, then per-launch CUDA events) and
    the perturb pass; main() turns each update line into a roofline report."""
    import torch
    import synthetic
    out = []
    N = table.numel

    def timed(fn, reps):
        fn()
        ev = []
        for _ in range(reps):
            x0, x1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            x0.record(stream)
            fn()
            x1.record(stream)
            ev.append((x0, x1))
        torch.cuda.synchronize()
        return [x0.elapsed_time(x1) for x0, x1 in ev]

    for K in [int(k) for k in a.sweep.split(",") if k]:
        seeds = jb.seeds_array([(int(m), 7, 0) for m in synthetic.machine_ids(K, 910)])
        q = synthetic.byte_codes(K, 910)
        reps = SWEEP_REPS.get(K, 3)
        ms = timed(lambda: jb.jb_apply_updates(table, seeds, q, a.lr, 1.0, a.qscale, stream), reps)
        out.append({"K": K, "ms": ms})
    pms = timed(lambda: jb.jb_perturb(table, (1, 2, 3), a.eps, stream), 20)
    st = stats(pms)
    es = table.tensors[0].element_size()
    out.append({"perturb_ms": st["mean"], "perturb_ms_best": st["best"], "perturb_ms_median": st["median"],
                "param_seed_per_s": N / (st["best"] / 1e3),
                "hbm_gbs": 2 * es * N / (st["best"] / 1e3) / 1e9})
    nxt = []
    if a.next_legs:
        nxt.extend(next_legs(a, jb, table, stream))
        nxt.append(checksum_leg(jb, table, stream))
        nxt.append(q4_leg(a, jb, stream))
    if a.sweep_out:
        with open(a.sweep_out, "w") as f:
            for ln in out + nxt:
                f.write(json.dumps(ln) + "\n")
    return out, nxt


def next_legs(a, jb, table, stream):
    """The update from the weight backup (restore fused) against copy + update, and
    a replay of T steps against T separate updates, on the benchmark's set."""
    import torch
    import synthetic
    out = []
    ev = lambda: torch.cuda.Event(enable_timing=True)
    backup = jb.ParamTable([torch.empty_like(t) for t in table.tensors], table.flat_offsets)
    for b, t in zip(backup.tensors, table.tensors):
        b.copy_(t)
    for K in sorted({1, 4, a.K}):
        seeds = jb.seeds_array([(int(m), 9, 0) for m in synthetic.machine_ids(K, 920)])
        q = synthetic.byte_codes(K, 920)
        for mode in ("copy+update", "fused", "fused+refresh"):
            def once():
                if mode == "copy+update":
                    for b, t in zip(backup.tensors, table.tensors):
                        t.copy_(b)
                    jb.jb_apply_updates(table, seeds, q, a.lr, 1.0, a.qscale, stream)
                else:
                    jb.jb_apply_updates_from(backup, table, seeds, q, a.lr, 1.0, a.qscale,
                                             write_src=(mode == "fused+refresh"), stream=stream)
            once()
            x0, x1 = ev(), ev()
            x0.record(stream)
            for _ in range(2):
                once()
            x1.record(stream)
            torch.cuda.synchronize()
            out.append({"leg": "restore+update", "mode": mode, "K": K, "ms": x0.elapsed_time(x1) / 2})
    del backup
    for T, Kt in ((16, 4), (64, 1)):
        steps = []
        for t in range(T):
            sd = jb.seeds_array([(int(m), 100 + t, 0) for m in synthetic.machine_ids(Kt, 930, t)])
            steps.append((sd, synthetic.byte_codes(Kt, 930, t), a.lr, float(Kt)))
        for mode in ("sequential", "replay"):
            def once():
                if mode == "replay":
                    jb.jb_replay_updates(table, steps, a.qscale, stream)
                else:
                    for sd, qq, lr, den in steps:
                        jb.jb_apply_updates(table, sd, qq, lr, den, a.qscale, stream)
            once()
            x0, x1 = ev(), ev()
            x0.record(stream)
            once()
            x1.record(stream)
            torch.cuda.synchronize()
            out.append({"leg": "replay", "mode": mode, "steps": T, "K_per_step": Kt,
                        "ms": x0.elapsed_time(x1),
                        "param_seed_per_s": table.numel * T * Kt / (x0.elapsed_time(x1) / 1e3)})
    return out


def checksum_leg(jb, table, stream):
    """The model checksum (ChecksumMatch): one read of theta, HBM-bound."""
    import torch
    out = torch.zeros(1, dtype=torch.int64, device="cuda")
    jb.jb_checksum(table, out, stream)
    x0, x1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    reps = 5
    x0.record(stream)
    for _ in range(reps):
        jb.jb_checksum(table, out, stream)
    x1.record(stream)
    torch.cuda.synchronize()
    ms = x0.elapsed_time(x1) / reps
    nbytes = table.numel * table.tensors[0].element_size()
    return {"leg": "checksum", "ms": ms, "bytes": nbytes, "hbm_gbs": nbytes / (ms / 1e3) / 1e9}


def q4_leg(a, jb, stream):
    """PerturbParameters on the benchmark's set stored as 4-bit weights (codes and
    64-element scales, synthetic values), one pass read + write."""
    import torch
    import synthetic
    specs = synthetic.opt_tensors(a.model)
    g = torch.Generator(device="cuda")
    g.manual_seed(synthetic.MASTER_SEED)
    tensors = []
    for sp in specs:
        n = sp.numel
        codes = torch.randint(0, 256, ((n + 1) // 2 + 8,), dtype=torch.uint8, device="cuda",
                              generator=g)
        scale = torch.rand(((n + 63) // 64,), device="cuda", generator=g) * 0.05
        tensors.append((codes, scale, n))
    table = jb.Q4Table(tensors)
    jb.jb_perturb_q4(table, (1, 2, 3), a.eps, stream)
    x0, x1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    x0.record(stream)
    for i in range(3):
        jb.jb_perturb_q4(table, (1, 2, 3), a.eps if i % 2 == 0 else -a.eps, stream)
    x1.record(stream)
    torch.cuda.synchronize()
    ms = x0.elapsed_time(x1) / 3
    n = sum(sp.numel for sp in specs)
    nbytes = 2 * sum((sp.numel + 1) // 2 + 4 * ((sp.numel + 63) // 64) for sp in specs)
    del tensors, table
    torch.cuda.empty_cache()
    return {"leg": "perturb_q4", "ms": ms, "param_seed_per_s": n / (ms / 1e3),
            "hbm_gbs": nbytes / (ms / 1e3) / 1e9}


if __name__ == "__main__":
    main()
