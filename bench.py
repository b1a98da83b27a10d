#!/usr/bin/env python
"""Masked decode-step throughput of the DOMINO hot path on GB300.

One step = one domino_step_decode call over one batch (Alg. 1): C.mask() with
v' = m (.) v and the greedy decode folded into it, then C.update() in the same
call's per-row merge.  Default workload: random
sparse DFA (Q = 5000, 32 byte classes), V = 128256, batch 256, bf16 logits
N(0, 3), rotating over enough logits buffers to exceed twice the L2.

Prints ONE JSON line (rank 0).  Metric = token-checks/s (batch x vocabulary
per second of whole decode steps); masked decode steps/s and per-kernel
rooflines are extra keys.

  python bench.py [--gpus N] [--steps K] [--warmup W] [--workload 3]
  python bench.py --impl reference ...   # the CPU oracle on host cores
"""
from __future__ import annotations

import argparse
import ctypes
import json
import math
import os
import statistics
import subprocess
import sys
import threading
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "token-checks/s and masked decode steps/s at 1 GB300; mask+logits HBM GB/s vs peak"
UNIT = "token-checks/s"
L2_BYTES = 129 * 1024 * 1024
WORKLOAD_HELP = {1: "kv16_v1024_b1", 2: "kv200_v32000_b32", 3: "sparse5000_v128256_b256",
                 4: "precompute_sparse20000_v128256", 5: "json300_pda_v152064_b128"}


def parse():
    p = argparse.ArgumentParser()
    p.add_argument("--gpus", type=int, default=1)
    p.add_argument("--steps", type=int, default=2000)
    p.add_argument("--warmup", type=int, default=5)
    p.add_argument("--impl", choices=["domino", "reference"], default="domino")
    p.add_argument("--workload", type=int, default=3, choices=sorted(WORKLOAD_HELP))
    p.add_argument("--e2e-steps", type=int, default=100)
    p.add_argument("--no-cpu-baseline", action="store_true")
    p.add_argument("--no-graph", action="store_true", help="launch eagerly (used for ncu launch lists)")
    p.add_argument("--cpu-seconds", type=float, default=12.0, help="target CPU time of the oracle baseline")
    return p.parse_args()


# ----------------------------------------------------------------------------
# distributed plumbing (replicas only: no data-path collective)
# ----------------------------------------------------------------------------
class Dist:
    def __init__(self):
        self.world = int(os.environ.get("WORLD_SIZE", "1"))
        self.rank = int(os.environ.get("RANK", "0"))
        self.local = int(os.environ.get("LOCAL_RANK", "0"))
        self.pg = None
        if self.world > 1:
            import torch.distributed as dist
            backend = "nccl" if _cuda_ok() else "gloo"
            dist.init_process_group(backend)
            self.pg = dist

    def barrier(self):
        if self.pg:
            self.pg.barrier()

    def max(self, x: float) -> float:
        if not self.pg:
            return x
        import torch
        dev = f"cuda:{self.local}" if _cuda_ok() and self.pg.get_backend() == "nccl" else "cpu"
        t = torch.tensor([x], dtype=torch.float64, device=dev)
        self.pg.all_reduce(t, op=self.pg.ReduceOp.MAX)
        return float(t.item())

    def close(self):
        if self.pg:
            self.pg.destroy_process_group()


def _cuda_ok():
    import torch
    return torch.cuda.is_available()


# ----------------------------------------------------------------------------
# SM clock / throttle sampling during the timed region (NVML, read only)
# ----------------------------------------------------------------------------
REASONS = {0x1: "gpu_idle", 0x2: "applications_clocks_setting", 0x4: "sw_power_cap", 0x8: "hw_slowdown",
           0x10: "sync_boost", 0x20: "sw_thermal_slowdown", 0x40: "hw_thermal_slowdown",
           0x80: "hw_power_brake_slowdown", 0x100: "display_clock_setting"}


class ClockSampler:
    def __init__(self, torch_dev: int, period_s: float = 0.001):
        self.period = period_s
        self.samples = []
        self.reasons = 0
        self.max_mhz = None
        self.ok = False
        self._stop = threading.Event()
        try:
            nv = ctypes.CDLL("libnvidia-ml.so.1")
            if nv.nvmlInit_v2() != 0:
                return
            h = ctypes.c_void_p()
            import torch
            uuid = None
            try:
                uuid = "GPU-" + str(torch.cuda.get_device_properties(torch_dev).uuid)
            except Exception:
                pass
            rc = nv.nvmlDeviceGetHandleByUUID(uuid.encode(), ctypes.byref(h)) if uuid else 1
            if rc != 0:
                vis = os.environ.get("CUDA_VISIBLE_DEVICES", "")
                idx = int(vis.split(",")[torch_dev]) if vis and vis.split(",")[0].isdigit() else torch_dev
                if nv.nvmlDeviceGetHandleByIndex_v2(idx, ctypes.byref(h)) != 0:
                    return
            self.nv, self.h = nv, h
            c = ctypes.c_uint()
            if nv.nvmlDeviceGetMaxClockInfo(h, 1, ctypes.byref(c)) == 0:
                self.max_mhz = c.value
            self._reason_fn = getattr(nv, "nvmlDeviceGetCurrentClocksEventReasons", None) or \
                getattr(nv, "nvmlDeviceGetCurrentClocksThrottleReasons")
            self.ok = True
        except Exception:
            self.ok = False

    def _run(self):
        c = ctypes.c_uint()
        r = ctypes.c_ulonglong()
        while not self._stop.is_set():
            if self.nv.nvmlDeviceGetClockInfo(self.h, 1, ctypes.byref(c)) == 0:
                self.samples.append(c.value)
            if self._reason_fn(self.h, ctypes.byref(r)) == 0:
                self.reasons |= r.value & ~0x1
            time.sleep(self.period)

    def start(self):
        """Samples until stop(); may be started again (the samples accumulate)."""
        if self.ok:
            self._stop = threading.Event()
            self._t = threading.Thread(target=self._run, daemon=True)
            self._t.start()

    def stop(self):
        if self.ok:
            self._stop.set()
            self._t.join()

    def summary(self, first: int = 0):
        """Median SM clock and the throttle reasons seen; `first`: the samples
        of the headline timed region (the region sampled first)."""
        if not self.ok or not self.samples:
            return {"sm_mhz": None, "sm_max_mhz": self.max_mhz, "reasons": ["unavailable"]}
        names = [n for bit, n in REASONS.items() if self.reasons & bit]
        out = {"sm_mhz": statistics.median(self.samples), "sm_max_mhz": self.max_mhz, "reasons": names,
               "samples": len(self.samples)}
        if first:
            out["timed_region_samples"] = first
            out["note"] = ("sampled every 1 ms during the timed steps and during every per-kernel timing "
                           "graph of this run")
        return out


def measured_peaks():
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            return json.load(f), "measured"
    except Exception:
        return {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0}, "fallback"


# ----------------------------------------------------------------------------
# CPU oracle baseline (bounded sample of the same workload)
# ----------------------------------------------------------------------------
def walk_stats(name: str):
    """Bytes the plain definition walks per check on this workload's trajectory,
    stored by tests/golden/make_walk_stats.py (None when not stored)."""
    p = os.path.join(ROOT, "tests", "golden", "walk_stats.json")
    try:
        with open(p) as f:
            return float(json.load(f)[name]["walk_steps_per_check_mean"])
    except (OSError, KeyError, ValueError):
        return None


def csrc_digest() -> str:
    """sha256 (first 16 hex digits) over the device sources, in name order."""
    import hashlib
    d = os.path.join(ROOT, "paper_2403_06988_gb300", "csrc")
    hs = hashlib.sha256()
    for fn in sorted(os.listdir(d)):
        if fn.endswith((".cu", ".cuh", ".h")):
            hs.update(fn.encode())
            with open(os.path.join(d, fn), "rb") as f:
                hs.update(f.read())
    return hs.hexdigest()[:16]


def ncu_traffic(name: str) -> dict:
    """DRAM bytes per launch (dram__bytes_read.sum + dram__bytes_write.sum) from
    the committed ncu summary, per kernel; a kernel whose source changed since
    the capture maps to None."""
    p = os.path.join(ROOT, "profiles", "traffic.json")
    try:
        with open(p) as f:
            rec = json.load(f)
        digest = csrc_digest()
    except (OSError, ValueError):
        return {}
    ent = rec.get("per_workload", {}).get(name, {})
    if ent.get("csrc_sha256_16") != digest:
        return {}
    return dict(ent.get("per_launch_bytes", {}))


def cpu_cores() -> int:
    try:
        return len(os.sched_getaffinity(0))
    except Exception:
        return os.cpu_count() or 1


def oracle_step_sample(w, P, states, stacks, rows, step, cores):
    """One oracle decode step (mask -> masked argmax/lse -> advance) on `rows` rows."""
    import oracle
    lg = w.logits(step, batch=rows)           # same values as the first `rows` rows
    st = states[:rows]
    sk = stacks[:rows] if w.automaton.rules is not None else None
    m, _, _ = P.step_mask(st, sk, n_threads=cores)
    arg, _, _ = oracle.mask_logits(lg, m, want_logprobs=w.want_logprobs, n_threads=cores)
    P.advance(st, sk, arg, w.automaton.start)


def cpu_baseline(w, target_s: float):
    import oracle
    cores = cpu_cores()
    P = oracle.Problem.from_workload(w)
    states, stacks = w.initial_configs()
    V = w.vocab.n_tokens
    rows = min(w.batch, max(1, cores))
    t0 = time.perf_counter()
    oracle_step_sample(w, P, states, stacks, rows, 0, cores)
    t1 = time.perf_counter() - t0
    reps = max(1, int(target_s / max(t1, 1e-3)))
    # logits generation is not part of the oracle's work: pre-generate
    lgs = [w.logits(i, batch=rows) for i in range(min(reps, 4))]
    t0 = time.perf_counter()
    for r in range(reps):
        lg = lgs[r % len(lgs)]
        st = states[:rows]
        sk = stacks[:rows] if w.automaton.rules is not None else None
        m, _, _ = P.step_mask(st, sk, n_threads=cores)
        arg, _, _ = oracle.mask_logits(lg, m, want_logprobs=w.want_logprobs, n_threads=cores)
        P.advance(st, sk, arg, w.automaton.start)
    dt = time.perf_counter() - t0
    # the same step on one core: a quarter of the time budget
    lg1 = w.logits(0, batch=1)
    sk1 = stacks[:1] if w.automaton.rules is not None else None
    reps1, t0 = 0, time.perf_counter()
    while True:
        m, _, _ = P.step_mask(states[:1], sk1, n_threads=1)
        arg, _, _ = oracle.mask_logits(lg1, m, want_logprobs=w.want_logprobs, n_threads=1)
        P.advance(states[:1], sk1, arg, w.automaton.start)
        reps1 += 1
        dt1 = time.perf_counter() - t0
        if dt1 > target_s / 4:
            break
    return {"value": rows * V * reps / dt, "unit": UNIT, "cores": cores, "kind": "oracle",
            "sample": f"{reps} decode steps of {rows} of the {w.batch} rows (full vocabulary V={V}); "
                      f"step_mask + mask_logits + advance, OpenMP over rows",
            "steps_per_s_equiv": reps * rows / w.batch / dt,
            "single_thread": {"value": V * reps1 / dt1, "unit": UNIT, "cores": 1,
                              "sample": f"{reps1} decode steps of one row"}}


# ----------------------------------------------------------------------------
# reference arm: the oracle timed on the host cores
# ----------------------------------------------------------------------------
def run_reference(args, dist: Dist):
    from paper_2403_06988_gb300 import synth
    if dist.rank != 0:
        return
    import oracle
    w = synth.workload(args.workload)
    cores = cpu_cores()
    P = oracle.Problem.from_workload(w)
    if w.config == 4:
        return run_reference_precompute(args, w, P, cores)
    states, stacks = w.initial_configs()
    V = w.vocab.n_tokens
    rows = min(w.batch, max(1, cores))
    # size each step's sample so that K + W steps stay within about two minutes
    t0 = time.perf_counter()
    oracle_step_sample(w, P, states, stacks, rows, 0, cores)
    per = time.perf_counter() - t0
    budget = 120.0 / max(1, args.steps + args.warmup)
    rows = max(1, min(rows, int(rows * budget / max(per, 1e-4))))
    for i in range(args.warmup):
        oracle_step_sample(w, P, states, stacks, rows, i, cores)
    lgs = [w.logits(i, batch=rows) for i in range(4)]
    t0 = time.perf_counter()
    for i in range(args.steps):
        st = states[:rows]
        sk = stacks[:rows] if w.automaton.rules is not None else None
        m, _, _ = P.step_mask(st, sk, n_threads=cores)
        arg, _, _ = oracle.mask_logits(lgs[i % 4], m, want_logprobs=w.want_logprobs, n_threads=cores)
        P.advance(st, sk, arg, w.automaton.start)
    dt = time.perf_counter() - t0
    value = rows * V * args.steps / dt
    line = {"impl": "reference", "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": args.gpus,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": dt * 1e3 / args.steps,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
            "data": "synthetic", "config": {"workload": w.name, "batch": w.batch, "vocab": V,
                                            "states": w.automaton.n_states, "sample_rows_per_step": rows},
            "cpu_baseline": {"value": value, "unit": UNIT, "cores": cores, "kind": "oracle",
                             "sample": f"{rows} of {w.batch} rows per step, full vocabulary"},
            "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)


def precompute_sample(w, P, rows: int, cores: int, step: int = 0):
    """The oracle's state x token table for `rows` states (next states and mask)."""
    Q = w.automaton.n_states
    states = ((np.arange(rows, dtype=np.int64) * 7919 + step * rows) % Q).astype(np.int32)
    P.step_mask(states, None, want_next=True, n_threads=cores)


def cpu_baseline_precompute(w, target_s: float):
    import oracle
    cores = cpu_cores()
    P = oracle.Problem.from_workload(w)
    rows = max(1, cores)
    t0 = time.perf_counter()
    precompute_sample(w, P, rows, cores)
    reps = max(1, int(target_s / max(time.perf_counter() - t0, 1e-3)))
    t0 = time.perf_counter()
    for r in range(reps):
        precompute_sample(w, P, rows, cores, r + 1)
    dt = time.perf_counter() - t0
    return {"value": rows * w.vocab.n_tokens * reps / dt, "unit": UNIT, "cores": cores, "kind": "oracle",
            "sample": f"{reps} x {rows} of the {w.automaton.n_states} table rows (next states + mask), "
                      f"OpenMP over rows"}


def run_reference_precompute(args, w, P, cores):
    V, Q = w.vocab.n_tokens, w.automaton.n_states
    rows = max(1, cores)
    t0 = time.perf_counter()
    precompute_sample(w, P, rows, cores)
    per = time.perf_counter() - t0
    budget = 120.0 / max(1, args.steps + args.warmup)
    rows = max(1, min(Q, int(rows * budget / max(per, 1e-4))))
    for i in range(args.warmup):
        precompute_sample(w, P, rows, cores, i)
    t0 = time.perf_counter()
    for i in range(args.steps):
        precompute_sample(w, P, rows, cores, i)
    dt = time.perf_counter() - t0
    value = rows * V * args.steps / dt
    line = {"impl": "reference", "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": args.gpus,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": dt * 1e3 / args.steps,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "int32",
            "data": "synthetic", "config": {"workload": w.name, "states": Q, "vocab": V,
                                            "sample_rows_per_step": rows},
            "cpu_baseline": {"value": value, "unit": UNIT, "cores": cores, "kind": "oracle",
                             "sample": f"{rows} of {Q} table rows per step, full vocabulary"},
            "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)


def run_precompute(args, dist: Dist):
    """Config 4: one step = the whole state x token table (next states int32 [Q][V] + mask)."""
    import torch

    from paper_2403_06988_gb300 import Domino, synth
    from paper_2403_06988_gb300 import _binding as B

    dev_id = dist.local
    torch.cuda.set_device(dev_id)
    dev = f"cuda:{dev_id}"
    w = synth.workload(4)
    d = Domino.from_parts(w.automaton, w.vocab, device=dev_id)
    info = d.info()
    Q, V, Wd = info["n_states"], info["n_tokens"], info["n_words"]
    nxt = torch.empty((Q, V), dtype=torch.int32, device=dev)
    mask = torch.empty((Q, Wd), dtype=torch.int32, device=dev)
    L, h = B.lib(), d.h
    p_n, p_m = nxt.data_ptr(), mask.data_ptr()
    s = torch.cuda.Stream(device=dev)
    K, Wm = args.steps, args.warmup

    def step(i, sp):
        if L.domino_precompute_table(h, p_n, p_m, sp):
            raise RuntimeError("precompute failed")
    with torch.cuda.stream(s):
        for i in range(Wm):
            step(i, s.cuda_stream)
    torch.cuda.synchronize()
    t0 = torch.cuda.Event(enable_timing=True)
    t1 = torch.cuda.Event(enable_timing=True)
    sampler = ClockSampler(dev_id)
    dist.barrier()
    torch.cuda.synchronize()
    sampler.start()
    with torch.cuda.stream(s):           # one launch per step, each far longer than a launch
        t0.record()
        for i in range(K):
            step(i, s.cuda_stream)
        t1.record()
    torch.cuda.synchronize()
    sampler.stop()
    dist.barrier()
    ms = dist.max(t0.elapsed_time(t1))
    if d.device_error():
        raise RuntimeError("device error word set")
    # end to end: the table computed and read back into pinned host memory
    host_n = torch.empty((Q, V), dtype=torch.int32).pin_memory()
    host_m = torch.empty((Q, Wd), dtype=torch.int32).pin_memory()
    Ke = max(1, min(2, K))
    e0 = torch.cuda.Event(enable_timing=True)
    e1 = torch.cuda.Event(enable_timing=True)
    dist.barrier()
    torch.cuda.synchronize()
    with torch.cuda.stream(s):
        e0.record()
        for i in range(Ke):
            step(i, s.cuda_stream)
            host_n.copy_(nxt, non_blocking=True)
            host_m.copy_(mask, non_blocking=True)
        e1.record()
    torch.cuda.synchronize()
    e2e_ms = dist.max(e0.elapsed_time(e1))
    n = dist.world
    out_bytes = Q * V * 4 + Q * Wd * 4
    t = ms / K / 1e3
    peaks, peak_kind = measured_peaks()
    hbm_peak = float(peaks.get("hbm_gbs", 6800.0))
    traffic = ncu_traffic(w.name)
    line = {
        "metric": METRIC, "value": n * Q * V * K / (ms / 1e3), "unit": UNIT, "n_gpus": n, "steps": K,
        "warmup": Wm, "ms_per_step": ms / K, "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
        "dtype": "int32", "data": "synthetic",
        "config": {"workload": w.name, "states": Q, "vocab": V, "byte_classes": info["n_classes"],
                   "table_in_smem": info["table_in_smem"], "output_bytes": out_bytes,
                   "l2": f"each step writes {out_bytes / 2**30:.1f} GiB (> L2)", "parallelism": f"replicas x{n}"},
        "roofline": {"kernel": "step_mask (row = state, next states written)", "bound": "hbm",
                     "achieved": out_bytes / t / 1e9, "peak": hbm_peak, "unit": "GB/s",
                     "frac": out_bytes / t / 1e9 / hbm_peak, "traffic": traffic.get("precompute"),
                     "algorithmic_units_per_launch": out_bytes, "peak_source": f"hbm_gbs {peak_kind}"},
        "e2e": {"value": n * Q * V * Ke / (e2e_ms / 1e3), "unit": UNIT, "h2d_bytes_per_step": 0,
                "d2h_bytes_per_step": out_bytes, "steps": Ke,
                "api": "domino_precompute_table + copy of the table to pinned host memory"},
        # the tree walk: tree_clear_kernel then tree_tile_kernel; else one step_kernel
        "gpu_launches": K * (2 if info["walk_tree"] else 1),
        "clocks": sampler.summary(),
    }
    if dist.rank == 0 and n == 1 and not args.no_cpu_baseline:
        line["cpu_baseline"] = cpu_baseline_precompute(w, args.cpu_seconds)
    if dist.rank == 0:
        print(json.dumps(line), flush=True)
    d.close()


# ----------------------------------------------------------------------------
# the GPU arm
# ----------------------------------------------------------------------------
def run_domino(args, dist: Dist):
    import torch

    from paper_2403_06988_gb300 import Domino, synth
    from paper_2403_06988_gb300 import _binding as B

    dev_id = dist.local
    torch.cuda.set_device(dev_id)
    dev = f"cuda:{dev_id}"
    w = synth.workload(args.workload)
    a, v = w.automaton, w.vocab
    d = Domino.from_parts(a, v, device=dev_id)
    info = d.info()
    Bsz, V, Wd = w.batch, v.n_tokens, info["n_words"]
    stack = a.rules is not None
    states0, stacks0 = w.initial_configs(part=2 + 17 * dist.rank)   # each replica its own batch
    states = torch.from_numpy(states0).to(dev)
    stacks = torch.from_numpy(stacks0.view(np.int64)).to(dev) if stack else None
    esz = 2 if w.logits_dtype == "bf16" else 4
    logit_bytes = Bsz * V * esz
    nbuf = max(4, math.ceil(2.2 * L2_BYTES / logit_bytes))
    host_logits = [w.logits(100 + i) for i in range(nbuf)]

    def to_dev(x):
        t = torch.from_numpy(x.view(np.int16) if x.dtype == np.uint16 else x).to(dev)
        return t.view(torch.bfloat16) if x.dtype == np.uint16 else t
    logits = [to_dev(x) for x in host_logits]
    mask = torch.empty((Bsz, Wd), dtype=torch.int32, device=dev)
    argmax = torch.empty(Bsz, dtype=torch.int32, device=dev)
    lse = torch.empty(Bsz, dtype=torch.float32, device=dev)
    logprobs = torch.empty((Bsz, V), dtype=torch.float32, device=dev) if w.want_logprobs else None
    dtype_code = B.DTYPE_BF16 if w.logits_dtype == "bf16" else B.DTYPE_F32
    L = B.lib()
    h = d.h
    # raw pointers once
    p_states, p_stacks = states.data_ptr(), (stacks.data_ptr() if stack else None)
    p_mask, p_arg, p_lse = mask.data_ptr(), argmax.data_ptr(), lse.data_ptr()
    p_lp = logprobs.data_ptr() if logprobs is not None else None
    p_logits = [t.data_ptr() for t in logits]
    # one step = one call. With the per-token walk and bf16 logits: the mask
    # step with the greedy decode folded in, then the per-row merge that also
    # advances each row. With the prefix-tree walk (two launches: clear, tree
    # tiles) or fp32 logits: mask step, logits pass, update. Plus the
    # log-probs pass where the workload asks for them.
    walk_launches = 2 if info.get("walk_tree") else 1
    fused = w.logits_dtype == "bf16" and not info.get("walk_tree")
    launches_per_step = (2 if fused else walk_launches + 2) + (1 if w.want_logprobs else 0)

    def step(i, stream_ptr):
        rc = L.domino_step_decode(h, p_states, p_stacks, Bsz, p_logits[i % nbuf], dtype_code, V, p_mask, p_arg, p_lse,
                                  p_lp, p_states, p_stacks, stream_ptr)
        if rc:
            raise RuntimeError(f"domino call failed ({rc})")

    K, Wm = args.steps, args.warmup
    n_world = dist.world
    s = torch.cuda.Stream(device=dev)
    with torch.cuda.stream(s):
        sp = s.cuda_stream
        for i in range(Wm):
            step(i, sp)
    torch.cuda.synchronize()

    def capture(n, body):
        """A CUDA graph of n calls of body(i, stream) on stream s (None: eager)."""
        if args.no_graph:
            return None
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g, stream=s, capture_error_mode="relaxed"):
            sp = torch.cuda.current_stream().cuda_stream
            for i in range(n):
                body(i, sp)
        g.replay()                          # upload + one untimed pass
        torch.cuda.synchronize()
        return g

    def timed(n, body, g, sampler=None, reps=1):
        """Device time (ms) of n calls (`reps` passes of them, averaged), events
        on the launching stream, synchronized on both sides."""
        t0 = torch.cuda.Event(enable_timing=True)
        t1 = torch.cuda.Event(enable_timing=True)
        dist.barrier()
        torch.cuda.synchronize()
        if sampler is not None:
            sampler.start()
        with torch.cuda.stream(s):
            t0.record()
            for _ in range(reps):
                if g is not None:
                    g.replay()
                else:
                    for i in range(n):
                        body(i, s.cuda_stream)
            t1.record()
        torch.cuda.synchronize()
        if sampler is not None:
            sampler.stop()
        dist.barrier()
        return t0.elapsed_time(t1) / reps

    def timed_long(n, body, g, sampler, min_ms=4.0):
        """timed() over enough passes of the graph to fill about min_ms of
        device time: steadier per-launch figures, and clock samples under load
        even when n is small."""
        est = timed(n, body, g)
        return timed(n, body, g, sampler, reps=max(1, min(200, math.ceil(min_ms / max(est, 1e-3)))))

    # ---- the timed region: K whole decode steps, nothing else in the graph ----
    graph = capture(K, step)
    sampler = ClockSampler(dev_id)   # also runs during the per-kernel graphs below
    ms = timed(K, step, graph, sampler)
    ms_max = dist.max(ms)
    first_samples = len(sampler.samples)
    err = d.device_error()
    if err:
        raise RuntimeError(f"device error word {err}")

    # ---- per-kernel average launch durations: each kernel alone, Kk launches
    # back to back in its own graph on the same stream (its inputs as in a step)
    Kk = min(K, 400)
    st_tmp = torch.empty_like(states)
    sk_tmp = torch.empty_like(stacks) if stack else None
    p_st_tmp, p_sk_tmp = st_tmp.data_ptr(), (sk_tmp.data_ptr() if stack else None)

    def k_step(i, sp):
        if L.domino_step_mask(h, p_states, p_stacks, Bsz, p_mask, None, sp):
            raise RuntimeError("step_mask failed")

    def k_logits(i, sp):
        if L.domino_mask_logits(h, p_logits[i % nbuf], dtype_code, Bsz, V, p_mask, p_arg, p_lse, p_lp, sp):
            raise RuntimeError("mask_logits failed")

    def k_fused(i, sp):
        if L.domino_step_decode(h, p_states, p_stacks, Bsz, p_logits[i % nbuf], dtype_code, V, p_mask, p_arg, p_lse,
                                p_lp, None, None, sp):
            raise RuntimeError("step_decode failed")

    def k_adv(i, sp):
        if L.domino_advance(h, p_states, p_stacks, p_arg, Bsz, p_st_tmp, p_sk_tmp, sp):
            raise RuntimeError("advance failed")
    def k_sample(i, sp):
        if L.domino_mask_sample(h, p_logits[i % nbuf], dtype_code, Bsz, V, p_mask, ctypes.c_float(1.0),
                                ctypes.c_uint64(0x5EED), ctypes.c_uint64(i), p_arg, sp):
            raise RuntimeError("mask_sample failed")
    # the other mask walk, on a second handle: the prefix tree (Alg. 2's
    # subterminal tree over byte classes) and the per-token walk each timed alone
    walk_kind = "prefix tree" if info.get("walk_tree") else "per token"
    os.environ["DOMINO_WALK"] = "token" if info.get("walk_tree") else "tree"
    d_other = Domino.from_parts(a, v, device=dev_id)
    del os.environ["DOMINO_WALK"]
    other_kind = "prefix tree" if d_other.info().get("walk_tree") else "per token"
    h_other = d_other.h

    def k_step_other(i, sp):
        if L.domino_step_mask(h_other, p_states, p_stacks, Bsz, p_mask, None, sp):
            raise RuntimeError("step_mask (other walk) failed")
    per_kernel = {}
    for name, body in (("step_mask", k_step), ("step_mask_other", k_step_other), ("mask_logits", k_logits),
                       ("step_decode", k_fused), ("advance", k_adv), ("mask_sample", k_sample)):
        g = capture(Kk, body)
        per_kernel[name] = dist.max(timed_long(Kk, body, g, sampler)) / Kk      # ms per launch
        del g
    if d_other.device_error():
        raise RuntimeError("device error in the other walk")
    d_other.close()
    if d.device_error():
        raise RuntimeError("device error after the per-kernel graphs")

    # ---- opportunistic masking on the same rows: the logits as generated
    # (random: most proposals are rejected) and an obedient model's logits
    # (+20 on every allowed token: proposals are accepted)
    scratch = torch.empty((Bsz, Wd), dtype=torch.int32, device=dev)
    n_fb = torch.zeros(1, dtype=torch.int32, device=dev)
    p_scr, p_nfb = scratch.data_ptr(), n_fb.data_ptr()

    def opp_body(bufs):
        def body(i, sp):
            if L.domino_opportunistic_step(h, bufs[i % len(bufs)], dtype_code, Bsz, V, p_states, p_stacks, p_scr,
                                           p_arg, p_nfb, sp):
                raise RuntimeError("opportunistic step failed")
        return body
    with torch.cuda.stream(s):
        L.domino_step_mask(h, p_states, p_stacks, Bsz, p_mask, None, s.cuda_stream)
    torch.cuda.synchronize()
    bits = ((mask.view(torch.int32).unsqueeze(-1) >> torch.arange(32, device=dev, dtype=torch.int32)) & 1)
    bits = bits.reshape(Bsz, Wd * 32)[:, :V].to(torch.float32)
    obedient = [(t.to(torch.float32) + 20.0 * bits).to(t.dtype).contiguous() for t in logits]
    del bits
    opportunistic = {}
    for name, bufs in (("random_logits", p_logits), ("obedient_logits", [t.data_ptr() for t in obedient])):
        body = opp_body(bufs)
        with torch.cuda.stream(s):
            body(0, s.cuda_stream)
        torch.cuda.synchronize()
        g = capture(Kk, body)
        ms_o = dist.max(timed_long(Kk, body, g, sampler))
        del g
        opportunistic[name] = {"us": ms_o / Kk * 1e3, "fallback_rows": int(n_fb.item()), "rows": Bsz}
    opportunistic["masked_greedy_us"] = per_kernel["step_decode"] * 1e3
    opportunistic["note"] = ("same rows, fixed states; tokens equal the masked greedy decode; obedient = +20 on "
                             "every allowed logit")
    del obedient, scratch
    if d.device_error():
        raise RuntimeError("device error in the opportunistic step")

    # ---- count-based speculation: the model's update, s = 4 proposals and the
    # acceptance, each alone (the verification is step_mask + mask_logits over
    # batch x (s + 1) configurations, the kernels timed above)
    n_keys = info["n_states"] * (3 if stack else 1)
    S_SPEC = 4
    counts = torch.zeros((n_keys, V), dtype=torch.int32, device=dev)
    best = torch.zeros(n_keys, dtype=torch.int64, device=dev)
    reached = torch.zeros(n_keys, dtype=torch.int32, device=dev)
    prop = torch.empty((Bsz, S_SPEC), dtype=torch.int32, device=dev)
    n_prop = torch.empty(Bsz, dtype=torch.int32, device=dev)
    chain_s = torch.empty((Bsz, S_SPEC + 1), dtype=torch.int32, device=dev)
    chain_k = torch.empty((Bsz, S_SPEC + 1), dtype=torch.int64, device=dev) if stack else None
    decoded = torch.zeros((Bsz, S_SPEC + 1), dtype=torch.int32, device=dev)
    n_acc = torch.empty(Bsz, dtype=torch.int32, device=dev)
    pc, pb, pr = counts.data_ptr(), best.data_ptr(), reached.data_ptr()
    pp, pn, pcs = prop.data_ptr(), n_prop.data_ptr(), chain_s.data_ptr()
    pck = chain_k.data_ptr() if stack else None

    def k_spec_update(i, sp):
        if L.domino_spec_update(h, pc, pb, pr, p_states, p_stacks, p_arg, Bsz, sp):
            raise RuntimeError("spec_update failed")

    def k_spec_propose(i, sp):
        if L.domino_spec_propose(h, pb, pr, p_states, p_stacks, Bsz, S_SPEC, 0, pp, pn, pcs, pck, sp):
            raise RuntimeError("spec_propose failed")

    def k_spec_accept(i, sp):
        if L.domino_spec_accept(h, pp, pn, decoded.data_ptr(), pcs, pck, Bsz, S_SPEC, n_acc.data_ptr(), None, None,
                                None, sp):
            raise RuntimeError("spec_accept failed")
    spec = {}
    for name, body in (("update", k_spec_update), ("propose_s4", k_spec_propose), ("accept", k_spec_accept)):
        with torch.cuda.stream(s):
            body(0, s.cuda_stream)
        torch.cuda.synchronize()
        g = capture(Kk, body)
        spec[name + "_us"] = dist.max(timed_long(Kk, body, g, sampler)) / Kk * 1e3
        del g
    spec["proposals_per_row"] = float(n_prop.float().mean().item())
    spec["count_table_bytes"] = n_keys * V * 4
    del counts
    if d.device_error():
        raise RuntimeError("device error in the speculation kernels")

    # ---- table-driven step (DFA only): masks and next states precomputed once
    # for every state, then per step a mask-row lookup fused into the logits
    # pass and one table read per sequence for the update
    table_step = None
    if not stack:
        Q = info["n_states"]
        t_next = torch.empty((Q, V), dtype=torch.int32, device=dev)
        t_mask = torch.empty((Q, Wd), dtype=torch.int32, device=dev)
        p_tn, p_tm = t_next.data_ptr(), t_mask.data_ptr()
        pc0 = torch.cuda.Event(enable_timing=True)
        pc1 = torch.cuda.Event(enable_timing=True)
        with torch.cuda.stream(s):
            L.domino_precompute_table(h, p_tn, p_tm, s.cuda_stream)   # warm
            pc0.record()
            if L.domino_precompute_table(h, p_tn, p_tm, s.cuda_stream):
                raise RuntimeError("precompute failed")
            pc1.record()
        torch.cuda.synchronize()
        st_tab = torch.from_numpy(states0).to(dev)
        p_st_tab = st_tab.data_ptr()

        def t_step(i, sp):
            rc = L.domino_mask_logits_table(h, p_logits[i % nbuf], dtype_code, Bsz, V, p_tm, p_st_tab, p_arg, p_lse,
                                            p_lp, sp)
            rc |= L.domino_advance_table(h, p_tn, p_st_tab, p_arg, Bsz, p_st_tab, sp)
            if rc:
                raise RuntimeError(f"table step failed ({rc})")
        with torch.cuda.stream(s):
            for i in range(Wm):
                t_step(i, s.cuda_stream)
        torch.cuda.synchronize()
        g = capture(K, t_step)
        ms_t = dist.max(timed_long(K, t_step, g, sampler))
        del g
        if d.device_error():
            raise RuntimeError("device error in the table-driven step")
        table_step = {"ms_per_step": ms_t / K, "token_checks_per_s": n_world * Bsz * V * K / (ms_t / 1e3),
                      "masked_decode_steps_per_s": n_world * K / (ms_t / 1e3),
                      "precompute_ms": pc0.elapsed_time(pc1), "table_bytes": Q * V * 4 + Q * Wd * 4,
                      "note": "mask rows looked up from the precomputed [Q][W] table inside the logits pass; "
                              "update = one read of next[s][t]"}
        del t_next, t_mask

    # ---- end to end through the host-buffer C entry point -------------------
    Ke = max(3, min(args.e2e_steps, K))
    pin = [torch.from_numpy(x.view(np.int16) if x.dtype == np.uint16 else x).pin_memory() for x in host_logits[:2]]
    st_h = torch.from_numpy(states0.copy()).pin_memory()
    sk_h = torch.from_numpy(stacks0.view(np.int64).copy()).pin_memory() if stack else None
    tok_h = torch.empty(Bsz, dtype=torch.int32).pin_memory()
    lse_h = torch.empty(Bsz, dtype=torch.float32).pin_memory()
    e_start = torch.cuda.Event(enable_timing=True)
    e_end = torch.cuda.Event(enable_timing=True)
    with torch.cuda.stream(s):
        sp = s.cuda_stream

        def e2e_step(i):
            rc = L.domino_decode_step_host(h, pin[i % 2].data_ptr(), dtype_code, Bsz, st_h.data_ptr(),
                                           sk_h.data_ptr() if stack else None, tok_h.data_ptr(), lse_h.data_ptr(),
                                           sp)
            if rc:
                raise RuntimeError(f"decode_step_host failed ({rc})")
        for i in range(8):   # warm-up: the handle times its two host paths on its first calls
            e2e_step(i)
        dist.barrier()
        torch.cuda.synchronize()
        e_start.record()
        for i in range(Ke):
            e2e_step(i)
        e_end.record()
    torch.cuda.synchronize()
    e2e_ms = dist.max(e_start.elapsed_time(e_end))
    h2d = logit_bytes + Bsz * 4 + (Bsz * 8 if stack else 0)
    d2h = Bsz * 4 * 3 + (Bsz * 8 if stack else 0)

    # ---- structure of the workload's masks: an untimed decode loop from the
    # same starting rows, counting allowed tokens and the rows that end (EOS
    # chosen, or nothing allowed) and so restart from the start state
    S = 32
    states.copy_(torch.from_numpy(states0).to(dev))
    if stack:
        stacks.copy_(torch.from_numpy(stacks0.view(np.int64)).to(dev))
    allowed = ends_eos = ends_dead = 0
    with torch.cuda.stream(s):
        for i in range(S):
            step(i, s.cuda_stream)
            s.synchronize()
            allowed += int(np.unpackbits(mask.cpu().numpy().view(np.uint8)).sum())
            am = argmax.cpu().numpy()
            ends_eos += int((am == v.eos_id).sum()) if v.eos_id >= 0 else 0
            ends_dead += int((am < 0).sum())
    torch.cuda.synchronize()
    structure = {"decode_steps": S, "allowed_fraction": allowed / (S * Bsz * V),
                 "allowed_per_row": allowed / (S * Bsz),
                 "resets_per_step": (ends_eos + ends_dead) / S, "eos_per_step": ends_eos / S,
                 "all_masked_per_step": ends_dead / S, "byte_classes": info["n_classes"],
                 "walk": walk_kind,
                 "note": "greedy decode from the bench's starting rows, counted from the mask and argmax outputs"}

    # ---- report ---------------------------------------------------------------
    n = dist.world
    value = n * Bsz * V * K / (ms_max / 1e3)
    peaks, peak_kind = measured_peaks()
    hbm_peak = float(peaks.get("hbm_gbs", 6800.0))
    walk = walk_stats(w.name)
    traffic = ncu_traffic(w.name)
    lg_bytes = Bsz * V * esz + Bsz * Wd * 4 + Bsz * 8 + (Bsz * V * 4 if w.want_logprobs else 0)
    t_ml = per_kernel["mask_logits"] * 1e-3
    t_sm = per_kernel["step_mask"] * 1e-3
    gbs = lg_bytes / t_ml / 1e9
    ml_dram = traffic.get("mask_logits")
    kernels = {
        "mask_logits": {"us": t_ml * 1e6, "algorithmic_bytes": lg_bytes, "gbs": gbs, "frac_hbm": gbs / hbm_peak,
                        "dram_bytes_ncu": ml_dram,
                        "dram_gbs": ml_dram / t_ml / 1e9 if ml_dram else None,
                        "frac_hbm_dram": ml_dram / t_ml / 1e9 / hbm_peak if ml_dram else None},
        "step_mask": {"us": t_sm * 1e6, "checks_per_s": Bsz * V / t_sm, "mask_bytes": Bsz * Wd * 4,
                      "dram_bytes_ncu": traffic.get("step_mask")},
        "step_decode": {"us": per_kernel["step_decode"] * 1e3,
                        "separate_us": (per_kernel["step_mask"] + per_kernel["mask_logits"]) * 1e3,
                        "dram_bytes_ncu": traffic.get("step_decode_fused") if fused else None,
                        "note": ("the timed step's mask + decode: the mask step folds the allowed logits of each "
                                 "tile (then a per-row merge; log-probs in one more pass where asked for)") if fused
                        else ("the timed step's mask + decode + update: the mask step, the logits pass, "
                              "then the update, back to back")},
        "advance": {"us": per_kernel["advance"] * 1e3},
        "mask_sample": {"us": per_kernel["mask_sample"] * 1e3,
                        "gbs": (lg_bytes - Bsz * V * 4 * w.want_logprobs - Bsz * 4) / (per_kernel["mask_sample"] * 1e-3)
                        / 1e9, "note": "Gumbel-max draw at T = 1 over the same masks (Philox per 4 allowed tokens)"},
        "timing": f"each kernel alone, {Kk} launches back to back in one CUDA graph replayed over about 4 ms, "
                  "events on its stream",
    }
    # transition-lookup peak: one conflict-free 32-lane shared-memory gather per
    # SM clock; every byte the definition walks is one table lookup
    sm_clk = float(peaks.get("sm_max_mhz", 2070.0)) * 1e6
    lookup_peak = torch.cuda.get_device_properties(dev_id).multi_processor_count * 32 * sm_clk / 1e9
    kernels["step_mask"]["walk"] = walk_kind
    kernels["step_mask_" + ("token" if info.get("walk_tree") else "tree")] = {
        "us": per_kernel["step_mask_other"] * 1e3, "walk": other_kind,
        "checks_per_s": Bsz * V / (per_kernel["step_mask_other"] * 1e-3)}
    if walk is not None:
        structure["walk_steps_per_check"] = walk
        trans = walk * Bsz * V
        kernels["step_mask"].update({"walk_steps_per_check": walk, "gtransitions_per_s": trans / t_sm / 1e9,
                                     "frac_lookup_peak": trans / t_sm / 1e9 / lookup_peak})
    if t_sm >= t_ml and walk is not None:
        roofline = {"kernel": "step_mask", "bound": "alu", "achieved": trans / t_sm / 1e9, "peak": lookup_peak,
                    "unit": "Gtransitions/s", "frac": trans / t_sm / 1e9 / lookup_peak,
                    "traffic": traffic.get("step_mask"), "algorithmic_units_per_launch": trans,
                    "peak_source": f"{lookup_peak:.0f} G lookups/s = SMs x 32 lanes x {sm_clk / 1e6:.0f} MHz",
                    "note": ("walk bound by shared-memory gathers and issue, not HBM; the mask step timed alone "
                             "(in the timed step the same kernel also folds the logits: kernels.step_decode)")
                    if fused else
                            ("the prefix-tree mask step (clear + tree-tile kernels, one call) timed alone as it runs "
                             "in the step; units are the lookups the plain per-token definition makes, of which "
                             "the tree walk makes fewer (shared prefixes walked once)")}
    else:
        roofline = {"kernel": "mask_logits", "bound": "hbm", "achieved": gbs, "peak": hbm_peak, "unit": "GB/s",
                    "frac": gbs / hbm_peak, "traffic": traffic.get("mask_logits"),
                    "algorithmic_units_per_launch": lg_bytes, "peak_source": f"hbm_gbs {peak_kind}"}
    line = {
        "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": n, "steps": K, "warmup": Wm,
        "ms_per_step": ms_max / K, "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
        "dtype": "int32+f32", "data": "synthetic",
        "config": {"workload": w.name, "batch": Bsz, "vocab": V, "states": a.n_states, "logits_dtype": w.logits_dtype,
                   "byte_classes": info["n_classes"], "table_in_smem": info["table_in_smem"],
                   "logprobs": w.want_logprobs,
                   "l2": f"logits rotate over {nbuf} buffers ({nbuf * logit_bytes / 2**20:.0f} MiB > 2x L2)",
                   "parallelism": f"replicas x{n}", "graph": graph is not None},
        "masked_decode_steps_per_s": n * K / (ms_max / 1e3),
        "structure": structure, "kernels": kernels, "roofline": roofline, "table_driven_step": table_step,
        "opportunistic": opportunistic, "speculation": spec,
        "e2e": {"value": n * Bsz * V * Ke / (e2e_ms / 1e3), "unit": UNIT, "h2d_bytes_per_step": h2d,
                "d2h_bytes_per_step": d2h, "steps": Ke, "api": "domino_decode_step_host with pinned host buffers",
                "h2d_note": "h2d_bytes_per_step counts the whole logits tensor; on the in-place path only the "
                            "allowed logits cross the link (the handle times both paths and uses the faster)"},
        "gpu_launches": K * launches_per_step,
        "gpu_launches_note": "timed region only; per-kernel graphs and e2e are timed separately",
        "clocks": sampler.summary(first_samples),
    }
    if dist.rank == 0 and n == 1 and not args.no_cpu_baseline:
        line["cpu_baseline"] = cpu_baseline(w, args.cpu_seconds)
    if dist.rank == 0:
        print(json.dumps(line), flush=True)
    d.close()


def main():
    args = parse()
    dist = Dist()
    try:
        if args.impl == "reference":
            run_reference(args, dist)
        elif args.workload == 4:
            run_precompute(args, dist)
        else:
            run_domino(args, dist)
    finally:
        dist.close()


if __name__ == "__main__":
    main()
