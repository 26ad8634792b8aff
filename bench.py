#!/usr/bin/env python3
"""Benchmark: one decode step of the paged KV path on the Llama-3-8B-shaped
layer (64 sequences, 32 query / 8 KV heads, head dim 128, block size 16,
lognormal context lengths with median 1024, sigma 1, clipped to 16384).

A step is the whole hot path for one batch: the host sequence table advances
every sequence by one token (growing reservations where needed) and syncs the
lengths and changed table entries to the device, then the new K/V rows are
appended and paged decode attention runs; by default the append is fused
into the attention pass (one attention kernel + the split-K combine).  The headline
value is algorithmic HBM GB/s of the step: K/V bytes read (each sequence's
whole context) + q read + output written + appended K/V written, divided by
the device time of the step.

Usage: python bench.py [--gpus N] [--steps K] [--warmup W] [--impl reference]
Prints one JSON line on rank 0.
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

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

METRIC = "paged decode-attn HBM GB/s (% of GB300 peak) and decode tokens/s at 1 GPU"
WORKLOAD = ("llama3-8b-layer: 64 seqs, 32 q / 8 kv heads, d=128, bs=16, bf16, lognormal context "
            "(median 1024, sigma 1, clip 16384), shuffled blocks, append + decode per step")


def load_peaks():
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            pk = json.load(f)
        return float(pk["hbm_gbs"]), "measured"
    except Exception:
        return 6800.0, "fallback"


class ClockSampler:
    """nvidia-smi clock/throttle samples while the timed region runs."""

    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index: int):
        self.gpu = gpu_index
        self.proc = None
        self.lines = []
        self.thread = None

    def start(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.gpu), f"--query-gpu={self.FIELDS}", "--format=csv,noheader,nounits",
                 "-lms", "100"], stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except Exception:
            self.proc = None
            return
        self.thread = threading.Thread(target=self._read, daemon=True)
        self.thread.start()

    def _read(self):
        for line in self.proc.stdout:
            self.lines.append(line.strip())

    def stop(self):
        if self.proc is None:
            return None
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except Exception:
            self.proc.kill()
        if self.thread:
            self.thread.join(timeout=2)
        sm, smax, reasons = [], 0.0, set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for ln in self.lines:
            parts = [p.strip() for p in ln.split(",")]
            if len(parts) < 9:
                continue
            try:
                sm.append(float(parts[1]))
                smax = max(smax, float(parts[2]))
            except ValueError:
                continue
            for nm, v in zip(names, parts[5:9]):
                if v.lower() == "active":
                    reasons.add(nm)
        if not sm:
            return None
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": smax, "reasons": sorted(reasons),
                "samples": len(sm)}


def algorithmic_bytes(b):
    kv = int(np.sum(b.ctx_lens.astype(np.int64))) * 2 * b.Hkv * b.d * 2
    q_out = 2 * b.S * b.Hq * b.d * 2
    app = 2 * b.S * b.Hkv * b.d * 2
    return kv, q_out, app


def oracle_baseline(b, budget_s: float):
    """Time the fp64 C oracle (single thread) on whole decode steps of the
    same workload (append + attention over every sequence) until budget_s
    elapses; return (GB/s of algorithmic bytes, steps, seconds)."""
    import oracle

    oracle.build()
    pool = b.pool
    lens = b.ctx_lens.copy()
    t0 = time.perf_counter()
    done_bytes = 0
    steps = 0
    while True:
        q, kn, vn = W_step_rows(b, steps)
        pool = oracle.append(pool, b.n_pages, b.page_elems, b.bs, b.Hkv, b.d, kn, vn, b.table, lens)
        oracle.paged_attention(pool, b.n_pages, b.page_elems, b.bs, b.Hkv, b.d, q, b.table, lens, b.scale)
        kv = int(lens.astype(np.int64).sum()) * 2 * b.Hkv * b.d * 2
        done_bytes += kv + 2 * b.S * b.Hq * b.d * 2 + 2 * b.S * b.Hkv * b.d * 2
        steps += 1
        lens = lens + 1
        el = time.perf_counter() - t0
        if el >= budget_s or steps >= 1000:
            return done_bytes / el / 1e9, steps, el


def W_step_rows(b, step):
    from paper_2606_12950_gb300 import workloads as W

    return W.step_rows(b.meta["seed"], step, b.S, b.Hq, b.Hkv, b.d)


def run_reference(args, rank, world):
    """The reference arm: the fp64 CPU oracle, timed on the host cores."""
    if rank != 0:
        return
    from paper_2606_12950_gb300 import workloads as W

    b = W.config2_llama8b()
    for i in range(args.warmup):
        oracle_baseline(b, 0.0)
    times = []
    total_bytes = 0
    for i in range(args.steps):
        gbs, steps, el = oracle_baseline(b, 0.0)
        times.append(el)
        total_bytes += gbs * el * 1e9
    t = sum(times)
    value = total_bytes / t / 1e9
    line = {
        "impl": "reference", "metric": METRIC, "value": value, "unit": "GB/s", "n_gpus": world,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": 1e3 * t / max(1, args.steps),
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
        "data": "synthetic", "config": {"workload": WORKLOAD, "S": b.S, "step": "one whole decode step"},
        "cpu_baseline": {"value": value, "unit": "GB/s", "cores": 1, "kind": "oracle",
                         "sample": "each step = one whole decode step (append + attention over all 64 "
                                   "sequences) of the same workload, single-threaded C fp64"},
        "e2e": {"value": value, "unit": "GB/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=100)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--num-splits", type=int, default=0)
    ap.add_argument("--variant", type=int, default=0, help="0 auto, 1 CUDA cores, 2 tensor-core MMA")
    ap.add_argument("--cpu-budget", type=float, default=10.0, help="seconds of oracle time for cpu_baseline")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--separate-append", action="store_true", help="append with its own kernel (unfused)")
    args = ap.parse_args()
    if args.warmup < 3 and args.impl == "ours":
        args.warmup = 3

    rank = int(os.environ.get("RANK", "0"))
    world = int(os.environ.get("WORLD_SIZE", "1"))
    local = int(os.environ.get("LOCAL_RANK", "0"))

    if args.impl == "reference":
        run_reference(args, rank, world)
        return

    import torch

    torch.cuda.set_device(local)
    dist = None
    if world > 1:
        import torch.distributed as dist

        dist.init_process_group("nccl", device_id=torch.device("cuda", local))

    from paper_2606_12950_gb300 import kvpool as K
    from paper_2606_12950_gb300 import workloads as W
    from paper_2606_12950_gb300.runner import DeviceBatch, DevicePool

    total_steps = 2 * (args.warmup + args.steps) + 8
    b = W.config2_llama8b(steps=max(100, total_steps))
    pool = DevicePool(b.n_pages, b.page_elems * 2, b.bs, [(b.Hkv, b.d)], shuffle_seed=b.meta["seed"])
    pool.upload(b.pool)
    if args.variant:
        pool.set_variant(args.variant)
    db = DeviceBatch(pool, 0, b, args.num_splits)
    stream = torch.cuda.current_stream()

    # host sequence table: each sequence reserves its whole run up front
    # (Eq. 2 with the true total length); blocks come from the shuffled pool
    seqtab = K.SeqTab(pool.handle, 0, b.S, b.max_blocks)
    pre = b.meta["pre_lens"].astype(np.int64)
    for s in range(b.S):
        seqtab.reserve(s, int(pre[s]) + total_steps)
        seqtab.set_len(s, int(pre[s]))
    done = [0]  # decode steps issued so far

    def step_bytes(j):
        """algorithmic bytes of decode step j: (attention call, whole step)"""
        n = pre + 1 + j
        kv = int(n.sum()) * 2 * b.Hkv * b.d * 2
        qo = 2 * b.S * b.Hq * b.d * 2
        return kv + qo, kv + qo + 2 * b.S * b.Hkv * b.d * 2

    def step(ev_pair=None):
        seqtab.advance()                         # host: every live sequence gains this step's token
        seqtab.sync(db.table, db.lens, stream)   # lengths (and any changed entries) to the device
        if ev_pair is not None:
            ev_pair[0].record(stream)
        if args.separate_append:
            db.append(stream)
            db.attend(stream=stream)
        else:
            db.append_attend(stream)             # append fused into the attention pass
        if ev_pair is not None:
            ev_pair[1].record(stream)
        done[0] += 1

    for i in range(args.warmup):
        step()
    torch.cuda.synchronize()
    if dist:
        dist.barrier()
    clocks = ClockSampler(local)
    clocks.start()
    time.sleep(0.3)
    evs = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(args.steps)]
    t_start = torch.cuda.Event(enable_timing=True)
    t_end = torch.cuda.Event(enable_timing=True)
    torch.cuda.synchronize()
    if dist:
        dist.barrier()
    first = done[0]
    t_start.record(stream)
    for i in range(args.steps):
        step(evs[i])
    t_end.record(stream)
    torch.cuda.synchronize()
    clk = clocks.stop()
    ms = t_start.elapsed_time(t_end)
    attn_ms = [a.elapsed_time(z) for a, z in evs]
    if dist:
        tt = torch.tensor([ms], device="cuda")
        dist.all_reduce(tt, op=dist.ReduceOp.MAX)
        ms = float(tt.item())
    err = pool.error(stream)

    attn_bytes = [step_bytes(first + i)[1] for i in range(args.steps)]  # the call also appends
    kv_total = sum(step_bytes(first + i)[1] for i in range(args.steps))
    gbs = kv_total / (ms * 1e-3) / 1e9 * world
    tokens_per_s = b.S * args.steps / (ms * 1e-3) * world
    attn_avg_ms = float(np.mean(attn_ms))
    attn_gbs = float(np.mean(attn_bytes)) / (attn_avg_ms * 1e-3) / 1e9
    peak, peak_kind = load_peaks()

    # end to end: q / k / v from pinned host memory, output back to host
    q_h = [torch.from_numpy(x.view(np.int16)).pin_memory() for x in W_step_rows(b, 0)]
    out_h = torch.empty(db.out.shape, dtype=torch.bfloat16).pin_memory()
    h2d = sum(int(t.numel()) * 2 for t in q_h) + b.S * 4
    d2h = out_h.numel() * 2

    def e2e_step():
        db.q.view(torch.int16).copy_(q_h[0], non_blocking=True)
        db.k_new.view(torch.int16).copy_(q_h[1], non_blocking=True)
        db.v_new.view(torch.int16).copy_(q_h[2], non_blocking=True)
        step()
        out_h.copy_(db.out, non_blocking=True)

    for i in range(3):
        e2e_step()
    torch.cuda.synchronize()
    e0 = torch.cuda.Event(enable_timing=True)
    e1 = torch.cuda.Event(enable_timing=True)
    first_e2e = done[0]
    e0.record(stream)
    for i in range(args.steps):
        e2e_step()
    e1.record(stream)
    torch.cuda.synchronize()
    e2e_total = sum(step_bytes(first_e2e + i)[1] for i in range(args.steps))
    e2e_ms = e0.elapsed_time(e1)
    e2e_gbs = e2e_total / (e2e_ms * 1e-3) / 1e9 * world

    cpu = None
    if rank == 0 and not args.no_cpu_baseline:
        v, nst, el = oracle_baseline(b, args.cpu_budget)
        cpu = {"value": v, "unit": "GB/s", "cores": 1, "kind": "oracle",
               "sample": f"{nst} whole decode steps (append + attention over all {b.S} sequences) of the same "
                         f"workload, single-threaded C fp64, {el:.1f} s"}

    traffic = None
    prof = os.path.join(ROOT, "profiles", "traffic.json")
    if os.path.exists(prof):
        try:
            with open(prof) as f:
                traffic = json.load(f).get("paged_attn_llama8b_bytes_per_launch")
        except Exception:
            traffic = None

    line = {
        "metric": METRIC, "value": gbs, "unit": "GB/s", "n_gpus": world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": ms / args.steps, "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "bf16", "data": "synthetic",
        "config": {"workload": WORKLOAD, "S": b.S, "Hq": b.Hq, "Hkv": b.Hkv, "d": b.d, "bs": b.bs,
                   "context_tokens_first_step": int((pre + 1 + first).sum()),
                   "kv_bytes_per_step": int(attn_bytes[0]), "l2": "inputs larger than L2 (no flush needed)",
                   "num_splits": args.num_splits, "variant": args.variant,
                   "parallelism": f"replicas x{world}" if world > 1 else "single GPU"},
        "decode_tokens_per_s": tokens_per_s,
        "roofline": {"bound": "hbm", "achieved": attn_gbs, "peak": peak, "unit": "GB/s",
                     "frac": attn_gbs / peak, "traffic": traffic, "kernel": "paged_attn_kernel",
                     "peak_kind": peak_kind, "attn_ms": attn_avg_ms},
        "step_frac_of_peak": gbs / world / peak,
        "e2e": {"value": e2e_gbs, "unit": "GB/s", "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h},
        "gpu_launches": (4 if args.separate_append else 3) * args.steps,
        "clocks": clk,
        "device_error": err,
        "cpu_baseline": cpu,
    }
    if rank == 0:
        print(json.dumps(line), flush=True)
    if dist:
        dist.barrier()
        dist.destroy_process_group()


if __name__ == "__main__":
    main()
