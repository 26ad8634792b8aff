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
import gc
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

    def start(self, cores=None):
        """cores: CPU set for the nvidia-smi child (default: this thread's)"""
        pre = (lambda: os.sched_setaffinity(0, cores)) if cores else None
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.gpu), f"--query-gpu={self.FIELDS}", "--format=csv,noheader,nounits",
                 "-lms", "100"], stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True, preexec_fn=pre)
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


def pin_process(local_rank: int):
    """Keep this process on four cores (a set per local rank), set before
    torch and the CUDA driver start their threads so that every thread
    created later inherits it.  With the submitting thread and the driver's
    threads free to spread over the cores, the step's launches reached the
    GPU late enough to cost the programmatic overlap of consecutive kernels
    (measured on a GB300 machine, config 2: 37 us of host time and 63 us per
    step unpinned, 23 us and 58.5 us pinned).  Returns the cores, or None."""
    try:
        allowed = sorted(os.sched_getaffinity(0))
    except (AttributeError, OSError):
        return None
    if len(allowed) < 8:
        return None
    cores = {allowed[(2 + 4 * local_rank + i) % len(allowed)] for i in range(4)}
    try:
        os.sched_setaffinity(0, cores)
    except OSError:
        return None
    return sorted(cores)


def aggregate_ranks(dist, device, ms: float, e2e_ms: float, units: dict) -> tuple:
    """Whole-job figures of N independent replicas: the slowest rank's time
    (max over ranks) and the units every rank processed (sum over ranks).
    With dist None (one process) the inputs come back unchanged."""
    if dist is None:
        return ms, e2e_ms, dict(units)
    import torch

    keys = sorted(units)
    t = torch.tensor([ms, e2e_ms], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    u = torch.tensor([float(units[k]) for k in keys], dtype=torch.float64, device=device)
    dist.all_reduce(u, op=dist.ReduceOp.SUM)
    tl, ul = t.tolist(), u.tolist()
    return tl[0], tl[1], dict(zip(keys, ul))


def oracle_lap_steps(b) -> int:
    """How many consecutive decode steps the batch's fixed table holds from
    its step-0 lengths: step i appends at position ctx_lens + i - 1, which
    must fall inside the blocks the table row lists.  At least 1."""
    cap = (b.table >= 0).sum(axis=1).astype(np.int64) * b.bs
    return max(1, int((cap - b.ctx_lens.astype(np.int64)).min()) + 1)


def _step_bytes(b, lens) -> int:
    kv = int(lens.astype(np.int64).sum()) * 2 * b.Hkv * b.d * 2
    return kv + 2 * b.S * b.Hq * b.d * 2 + 2 * b.S * b.Hkv * b.d * 2


def oracle_baseline(b, budget_s: float, max_steps: int = 1000):
    """Time the fp64 C oracle (single thread) on whole decode steps of the
    same workload (append + attention over every sequence) until budget_s
    elapses or max_steps steps are done; return (GB/s of algorithmic bytes,
    steps, seconds).  The steps run in laps of at most oracle_lap_steps(b):
    each lap starts again from the step-0 pool and lengths (untimed), so an
    append never leaves the table's reserved blocks however fast the host
    is, and the lengths follow the same schedule as the GPU arm's steps."""
    import oracle

    oracle.build()
    lap = oracle_lap_steps(b)
    el = 0.0
    done_bytes = 0
    steps = 0
    while True:
        pool = b.pool
        lens = b.ctx_lens.copy()
        for i in range(lap):
            t0 = time.perf_counter()
            q, kn, vn = W_step_rows(b, i)
            pool = oracle.append(pool, b.n_pages, b.page_elems, b.bs, b.Hkv, b.d, kn, vn, b.table, lens)
            oracle.paged_attention(pool, b.n_pages, b.page_elems, b.bs, b.Hkv, b.d, q, b.table, lens, b.scale)
            el += time.perf_counter() - t0
            done_bytes += _step_bytes(b, lens)
            steps += 1
            lens = lens + 1
            if el >= budget_s or steps >= max_steps:
                return done_bytes / el / 1e9, steps, el


def oracle_baseline_parallel(b, budget_s: float, cores, max_steps: int = 1000):
    """The same whole decode steps as oracle_baseline, with each step's
    attention spread over one thread per core: thread i computes the
    sequences at ranks i, i + T, ... of a longest-first order (the oracle's
    own seq_ids subset; ctypes releases the interpreter lock during the C
    call, so the threads run at once).  The append writes the pool in place
    (the oracle's inplace option) instead of into a fresh copy of it; the
    oracle's arithmetic is unchanged.  Laps as in oracle_baseline: between
    laps the pool is copied back from the step-0 pool outside the timed
    steps.  Returns (GB/s, steps, seconds, threads)."""
    from concurrent.futures import ThreadPoolExecutor

    import oracle

    oracle.build()
    T = max(1, len(cores))
    lap = oracle_lap_steps(b)
    order = np.argsort(-b.ctx_lens.astype(np.int64), kind="stable")
    subsets = [order[i::T].astype(np.int32) for i in range(T)]
    pool = np.array(b.pool, dtype=np.uint16, copy=True)  # appended in place below
    try:
        before = os.sched_getaffinity(0)
        os.sched_setaffinity(0, cores)  # threads created below inherit every core
    except (AttributeError, OSError):
        before = None
    try:
        with ThreadPoolExecutor(T) as ex:
            el = 0.0
            done_bytes = 0
            steps = 0
            finished = False
            while not finished:
                if steps:
                    np.copyto(pool, b.pool)  # back to the step-0 pool (untimed)
                lens = b.ctx_lens.copy()
                for i in range(lap):
                    t0 = time.perf_counter()
                    q, kn, vn = W_step_rows(b, i)
                    oracle.append(pool, b.n_pages, b.page_elems, b.bs, b.Hkv, b.d, kn, vn, b.table, lens,
                                  inplace=True)
                    outs = list(ex.map(lambda ids: oracle.paged_attention(pool, b.n_pages, b.page_elems, b.bs,
                                                                          b.Hkv, b.d, q, b.table, lens, b.scale,
                                                                          seq_ids=ids),
                                       subsets))
                    el += time.perf_counter() - t0
                    done_bytes += _step_bytes(b, lens)
                    steps += 1
                    lens = lens + 1
                    if el >= budget_s or steps >= max_steps:
                        finished = True
                        break
    finally:
        if before is not None:
            os.sched_setaffinity(0, before)
    # every sequence was computed by exactly one thread in the last step
    covered = sum((~np.isnan(o[:, 0, 0])).astype(np.int64) for o in outs)
    if not np.all(covered == 1):
        raise RuntimeError("threaded oracle baseline: the subsets do not cover the batch once")
    return done_bytes / el / 1e9, steps, el, T


def cpu_model() -> str:
    """The host CPU's model name (lscpu's, which names Arm cores too), else
    /proc/cpuinfo's first model line, else the platform's."""
    import subprocess

    try:
        out = subprocess.run(["lscpu"], capture_output=True, text=True, timeout=10).stdout
        for line in out.splitlines():
            if line.strip().lower().startswith("model name"):
                return line.split(":", 1)[1].strip()
    except (OSError, subprocess.SubprocessError):
        pass
    try:
        with open("/proc/cpuinfo") as f:
            for line in f:
                if line.lower().startswith(("model name", "cpu part", "hardware")):
                    return line.split(":", 1)[1].strip()
    except OSError:
        pass
    import platform

    return platform.processor() or platform.machine()


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


# ----------------------------------------------------------------- workloads
class Llama8B:
    """Config 2: every sequence reserves its whole run up front (Eq. 2 with the
    true total length); each step every sequence gains one token."""

    name = WORKLOAD

    def __init__(self, args, K, W, DevicePool, DeviceSteps):
        total = 2 * (args.warmup + args.steps) + 8
        b = W.config2_llama8b(steps=max(100, total))
        self.b = b
        vmm = getattr(args, "pool", "fixed") == "vmm"
        if vmm:
            # elastic pool: 4x the batch's need reserved as virtual memory,
            # chunks mapped as the reservations below allocate blocks
            from paper_2606_12950_gb300.runner import VmmPool

            self.pool = VmmPool(4 * b.n_pages * b.page_elems * 2, b.page_elems * 2, b.bs, [(b.Hkv, b.d)],
                                shuffle_seed=b.meta["seed"])
        else:
            self.pool = DevicePool(b.n_pages, b.page_elems * 2, b.bs, [(b.Hkv, b.d)], shuffle_seed=b.meta["seed"])
            self.pool.upload(b.pool)
        if args.variant:
            self.pool.set_variant(args.variant)
        self.tab = K.SeqTab(self.pool.handle, 0, b.S, b.max_blocks)
        self.pre = b.meta["pre_lens"].astype(np.int64)
        for s in range(b.S):
            self.tab.reserve(s, int(self.pre[s]) + total)
            self.tab.set_len(s, int(self.pre[s]))
        if vmm:
            table, _ = self.tab.host()
            self.pool.fill_random(np.unique(table[table >= 0]), b.meta["seed"])
        self.bufs = [DeviceSteps(self.pool, 0, b.S, b.S, b.Hq, b.Hkv, b.d, b.max_blocks, b.scale, b.q, b.k_new,
                                 b.v_new, args.num_splits)]
        self.S = b.S
        self.config = {"S": b.S, "Hq": b.Hq, "Hkv": b.Hkv, "d": b.d, "bs": b.bs,
                       "l2": "inputs larger than L2 (K+V ~ 326 MB per step; no flush needed)"}

    def host_step(self):
        self.tab.advance()
        n = self.tab.lens().astype(np.int64)
        kv = int(n.sum()) * 2 * self.b.Hkv * self.b.d * 2
        other = 2 * self.b.S * self.b.Hq * self.b.d * 2 + 2 * self.b.S * self.b.Hkv * self.b.d * 2
        return kv + other, kv + other  # (DRAM-algorithmic, logical) bytes

    def tables(self):
        return [(self.tab, self.bufs[0])]


class Chains:
    """Config 3: 256 Planner->Coder->Reviewer chains sharing a 2048-token
    prefix; the prefix is counted once per step for the DRAM roofline."""

    def __init__(self, args, K, W, DevicePool, DeviceSteps):
        from paper_2606_12950_gb300.schedules import AgentChains

        seed, n, d, Hq, Hkv, bs = 1003, 256, 128, 32, 8, 16
        self.name = ("agent-chains: 256 Planner->Coder->Reviewer chains, 32 q / 8 kv, d=128, bs=16, shared "
                     "2048-token prefix, stage outputs lognormal(300), reservations true x U[0.8,1.5]")
        max_blocks = (W.PREFIX_TOKENS + 4 * 4096 * 2) // bs + 8
        n_pages = 128 + n * 150 + 64
        page_elems = 2 * Hkv * bs * d
        host = np.empty(n_pages * page_elems, np.uint16)
        W.bf16_normal_fill(host, seed + 7919)
        self.pool = DevicePool(n_pages, page_elems * 2, bs, [(Hkv, d)], shuffle_seed=seed)
        self.pool.upload(host)
        del host
        if args.variant:
            self.pool.set_variant(args.variant)
        self.ch = AgentChains(self.pool.handle, 0, n, max_blocks, bs, seed)
        q, kn, vn = W.step_rows(seed, 0, n, Hq, Hkv, d)
        self.bufs = [DeviceSteps(self.pool, 0, n + 1, n, Hq, Hkv, d, max_blocks, d ** -0.5, q, kn, vn,
                                 args.num_splits)]
        self.S, self.Hq, self.Hkv, self.d = n, Hq, Hkv, d
        self.config = {"S": n, "Hq": Hq, "Hkv": Hkv, "d": d, "bs": bs,
                       "l2": "private K+V larger than L2; the 8.4 MB shared prefix is meant to hit in L2"}

    def host_step(self):
        self.ch.step()
        n = self.ch.ctx
        per_tok = 2 * self.Hkv * self.d * 2
        other = 2 * self.S * self.Hq * self.d * 2 + 2 * self.S * self.Hkv * self.d * 2
        unique = (int((n - W_PREFIX).sum()) + W_PREFIX) * per_tok
        logical = int(n.sum()) * per_tok
        return unique + other, logical + other

    def tables(self):
        return [(self.ch.tab, self.bufs[0])]

    def prefix_plan(self):
        return self.ch.prefix_plan()


class Coloc:
    """Config 4: three co-located layouts in one 90%-full pool; the same
    decode step (append + attention per layout) is repeated."""

    def __init__(self, args, K, W, DevicePool, DeviceSteps):
        self.name = ("co-location: 512 seqs over MHA 32/32, GQA 32/8, GQA 40/8 (d=128, bs=16) in one pool "
                     "filled to 90%, bounded Pareto(1.5) on [128, 32768]")
        batches, n_pages, page_elems = W.config4_colocation()
        self.pool = DevicePool(n_pages, page_elems * 2, 16, [(b.Hkv, b.d) for b in batches])
        self.pool.upload(batches[0].pool)
        if args.variant:
            self.pool.set_variant(args.variant)
        self.tabs, self.bufs = [], []
        for li, b in enumerate(batches):
            buf = DeviceSteps(self.pool, li, b.S, b.S, b.Hq, b.Hkv, b.d, b.max_blocks, b.scale, b.q, b.k_new,
                              b.v_new, args.num_splits)
            K.kv_block_table_upload(self.pool.handle, li, b.table, b.ctx_lens, buf.table, buf.lens)
            self.bufs.append(buf)
        only = getattr(args, "layout", None)
        if only is not None:
            # one co-located layout's batch alone, in the same 90%-full pool
            # (its per-layout figures; the step is then that batch's call)
            batches, self.bufs = [batches[only]], [self.bufs[only]]
            self.name += f"; layout {only} alone"
        self.batches = batches
        self.S = sum(b.S for b in batches)
        self.config = {"S": self.S, "layouts": [[b.Hq, b.Hkv, b.d] for b in batches], "bs": 16,
                       "pool_gb": n_pages * page_elems * 2 / 1e9, "l2": "inputs larger than L2"}

    def host_step(self):
        tot = 0
        for b in self.batches:
            tot += int(b.ctx_lens.astype(np.int64).sum()) * 2 * b.Hkv * b.d * 2
            tot += 2 * b.S * b.Hq * b.d * 2 + 2 * b.S * b.Hkv * b.d * 2
        return tot, tot

    def tables(self):
        return [(None, buf) for buf in self.bufs]


class LongCtx:
    """Config 5: 1024 heavy-tailed sequences that finish and are replaced."""

    def __init__(self, args, K, W, DevicePool, DeviceSteps):
        from paper_2606_12950_gb300.schedules import LongContextStress

        seed, S, d, Hq, Hkv, bs = 1005, 1024, 128, 32, 8, 32
        self.name = ("long-context stress: 1024 seqs, 32 q / 8 kv, d=128, bs=32, bounded Pareto(1.2) on "
                     "[256, 131072], sequences finish and are replaced")
        max_blocks = (131072 + 64) // bs + 2
        est = int(W.config5_lengths(np.random.default_rng(seed), S).sum())
        n_pages = int(1.4 * est / bs) + 4096
        page_elems = 2 * Hkv * bs * d
        self.pool = DevicePool(n_pages, page_elems * 2, bs, [(Hkv, d)], shuffle_seed=seed)
        # pool contents: seeded normal bf16 drawn on the device in one pass
        # (timing only; the parity tests use host-drawn pools)
        gen = __import__("torch").Generator(device="cuda").manual_seed(seed)
        self.pool.buf.view(__import__("torch").bfloat16).normal_(generator=gen)
        if args.variant:
            self.pool.set_variant(args.variant)
        self.lc = LongContextStress(self.pool.handle, 0, S, max_blocks, seed)
        q, kn, vn = W.step_rows(seed, 0, S, Hq, Hkv, d)
        self.bufs = [DeviceSteps(self.pool, 0, S, S, Hq, Hkv, d, max_blocks, d ** -0.5, q, kn, vn,
                                 args.num_splits)]
        self.S, self.Hq, self.Hkv, self.d = S, Hq, Hkv, d
        self.config = {"S": S, "Hq": Hq, "Hkv": Hkv, "d": d, "bs": bs, "l2": "inputs larger than L2"}

    def host_step(self):
        self.lc.step()
        n = self.lc.tab.lens().astype(np.int64)
        live = int((n > 0).sum())
        tot = int(n.sum()) * 2 * self.Hkv * self.d * 2 + 2 * live * self.Hq * self.d * 2 + \
            2 * live * self.Hkv * self.d * 2
        return tot, tot

    def tables(self):
        return [(self.lc.tab, self.bufs[0])]


W_PREFIX = 2048
WORKLOADS = {"llama8b": Llama8B, "chains": Chains, "coloc": Coloc, "longctx": LongCtx}


class StepRunner:
    """One decode step of a workload through the library's calls: the host
    bookkeeping, the table sync (carried by the decode launch when it fits),
    then append + attention per batch, by the call the options select."""

    def __init__(self, wl, args, K, stream):
        self.wl, self.args, self.K, self.stream = wl, args, K, stream
        self.launches_per_step = 0
        # a step's decode kernel may start while the previous step's combine
        # finishes (kv_set_attn_step_overlap)
        self.step_overlap = not getattr(args, "no_step_overlap", False)
        wl.pool.set_step_overlap(self.step_overlap)
        self.cascade = None
        if hasattr(wl, "prefix_plan") and not args.no_cascade and not args.separate_append:
            self.cascade = wl.prefix_plan()
            for _, buf in wl.tables():
                buf.use_cascade()
        self.fuse_sync = self.cascade is None and not args.separate_append and not args.separate_sync
        # shared prefix: the table sync rides in the kernel that writes the plan
        self.cascade_sync = self.cascade is not None and not args.separate_sync
        # co-located batches without host tables (the same step repeated): one call
        self.multi = (self.cascade is None and not args.separate_append and not args.separate_batches
                      and len(wl.tables()) > 1 and all(tab is None for tab, _ in wl.tables()))

    def sync_kernels(self):
        return sum(tab.counters()["sync_launches"] for tab, _ in self.wl.tables() if tab is not None)

    def step(self, ev_pair=None):
        """host bookkeeping, table sync, then append + attention per batch;
        returns the step's (DRAM-algorithmic, logical) bytes"""
        wl, args, K, stream = self.wl, self.args, self.K, self.stream
        nbytes = wl.host_step()
        n = 0
        if not self.fuse_sync and not self.cascade_sync:
            for tab, buf in wl.tables():
                if tab is not None:
                    tab.sync(buf.table, buf.lens, stream)
                    n += 1
        if ev_pair is not None:
            ev_pair[0].record(stream)
        if self.multi:
            # every batch's decode kernel as one chain, then the combines
            K.paged_decode_attn_multi(wl.pool.handle, [buf.batch() for _, buf in wl.tables()], stream)
            n += 2 * len(wl.tables())
        for tab, buf in (() if self.multi else wl.tables()):
            if self.fuse_sync and tab is not None:
                # table sync, append and attention: the decode launch carries
                # the sync when it fits (else a sync kernel runs first; those
                # launches are counted from the tables' counters)
                buf.sync_append_attend(tab, stream)
                n += 2
            elif self.cascade is not None:
                # plan (with the table sync when it fits), prefix kernel,
                # attention with the fused append, combine
                if self.cascade_sync:
                    buf.sync_cascade(tab, self.cascade, stream=stream)
                else:
                    buf.cascade(self.cascade, stream=stream)
                n += 4
            elif args.separate_append:
                buf.append(stream)
                buf.attend(stream)
                n += 3
            else:
                buf.append_attend(stream)  # the append fused into the attention pass
                n += 2
        if ev_pair is not None:
            ev_pair[1].record(stream)
        self.launches_per_step = n
        return nbytes


def measure_secondary(name, args, K, W, DevicePool, DeviceSteps, stream, peak):
    """The step of another workload (agent chains, co-location, long
    context), timed like the main one over min(steps, 30) steps after a
    short warm-up (device-resident inputs, CUDA events around the region);
    its buffers are freed afterwards."""
    import torch

    sargs = argparse.Namespace(**vars(args))
    sargs.workload = name
    wl = WORKLOADS[name](sargs, K, W, DevicePool, DeviceSteps)
    run = StepRunner(wl, sargs, K, stream)
    steps = max(1, min(args.steps, 30))
    gc.collect()
    gc.freeze()
    gc.disable()
    for _ in range(max(3, min(args.warmup, 5))):
        run.step()
    torch.cuda.synchronize()
    e0 = torch.cuda.Event(enable_timing=True)
    e1 = torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    nb = [run.step() for _ in range(steps)]
    e1.record(stream)
    torch.cuda.synchronize()
    ms = e0.elapsed_time(e1) / steps
    dram = sum(x[0] for x in nb) / steps
    logical = sum(x[1] for x in nb) / steps
    res = {"workload": wl.name, "steps": steps, "ms_per_step": ms, "gbs": dram / (ms * 1e-3) / 1e9,
           "frac_of_peak": dram / (ms * 1e-3) / 1e9 / peak, "decode_tokens_per_s": wl.S / (ms * 1e-3),
           "device_error": wl.pool.error(stream)}
    if logical != dram:
        res["logical_gbs"] = logical / (ms * 1e-3) / 1e9
    del run
    wl.pool.close()
    del wl
    gc.enable()
    gc.collect()
    torch.cuda.empty_cache()
    return res


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=100)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--workload", default="llama8b", choices=sorted(WORKLOADS))
    ap.add_argument("--num-splits", type=int, default=0)
    ap.add_argument("--variant", type=int, default=0, help="0 auto, 1 CUDA cores, 2 tensor-core MMA")
    ap.add_argument("--cpu-budget", type=float, default=10.0, help="seconds of oracle time for cpu_baseline")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-secondary", action="store_true",
                    help="llama8b: skip timing the agent-chains, co-location and long-context steps too")
    ap.add_argument("--separate-append", action="store_true", help="append with its own kernel (unfused)")
    ap.add_argument("--layout", type=int, default=None, choices=[0, 1, 2],
                    help="coloc: time one co-located layout's batch alone (0 MHA 32/32, 1 GQA 32/8, 2 GQA 40/8)")
    ap.add_argument("--separate-batches", action="store_true",
                    help="one call per co-located batch instead of one paged_decode_attn_multi call")
    ap.add_argument("--separate-sync", action="store_true",
                    help="table sync with its own kernel instead of carried by the decode (or plan) launch")
    ap.add_argument("--pool", default="fixed", choices=["fixed", "vmm"],
                    help="llama8b: a fixed device buffer, or the VMM-backed elastic pool")
    ap.add_argument("--no-step-overlap", action="store_true",
                    help="each step's decode kernel waits for the previous step's combine to complete first")
    ap.add_argument("--no-cascade", action="store_true",
                    help="agent chains: stream the shared prefix per chain instead of once per KV head")
    args = ap.parse_args()
    if args.warmup < 3 and args.impl == "ours":
        args.warmup = 3

    rank = int(os.environ.get("RANK", "0"))
    world = int(os.environ.get("WORLD_SIZE", "1"))
    local = int(os.environ.get("LOCAL_RANK", "0"))

    if args.impl == "reference":
        run_reference(args, rank, world)
        return

    try:
        all_cores = os.sched_getaffinity(0)
    except (AttributeError, OSError):
        all_cores = None
    pinned_cores = pin_process(local)  # before torch / CUDA create their threads
    import torch

    torch.cuda.set_device(local)
    dist = None
    if world > 1:
        import torch.distributed as dist

        dist.init_process_group("nccl", device_id=torch.device("cuda", local))

    from paper_2606_12950_gb300 import kvpool as K
    from paper_2606_12950_gb300 import workloads as W
    from paper_2606_12950_gb300.runner import DevicePool, DeviceSteps

    wl = WORKLOADS[args.workload](args, K, W, DevicePool, DeviceSteps)
    stream = torch.cuda.current_stream()
    runner = StepRunner(wl, args, K, stream)
    cascade, fuse_sync, multi = runner.cascade, runner.fuse_sync, runner.multi
    cascade_sync = runner.cascade_sync
    step, sync_kernels = runner.step, runner.sync_kernels

    # No garbage-collector pass inside the timed regions: a full pass over the
    # interpreter's objects (torch's included) stalled the submitting thread
    # for 3.4 ms in one measured step, long enough to drain the GPU's queue.
    # Everything alive now is moved out of the collector's view, and
    # collection is off until both timed regions are done.
    gc.collect()
    gc.freeze()
    gc.disable()

    # the clock sampler starts first; the warm-up steps then run right before
    # the timed region, so the GPU enters it busy rather than after an idle gap
    clocks = ClockSampler(local)
    clocks.start(cores=all_cores if pinned_cores else None)  # the sampler stays off the pinned cores' load
    time.sleep(0.3)
    for i in range(args.warmup):
        step()
    t_start = torch.cuda.Event(enable_timing=True)
    t_end = torch.cuda.Event(enable_timing=True)
    torch.cuda.synchronize()
    if dist:
        dist.barrier()
    step_bytes = []
    sync0 = sync_kernels()
    h0 = time.perf_counter()
    t_start.record(stream)
    for i in range(args.steps):
        step_bytes.append(step())
    t_end.record(stream)
    host_us = (time.perf_counter() - h0) * 1e6 / args.steps  # host submission time per step
    # sync kernels the calls launched themselves (syncs too large to carry)
    extra_sync_launches = sync_kernels() - sync0 if fuse_sync or cascade_sync else 0
    torch.cuda.synchronize()
    clk = clocks.stop()
    ms = t_start.elapsed_time(t_end)
    err = wl.pool.error(stream)

    dram_rank = sum(x[0] for x in step_bytes)
    logical_rank = sum(x[1] for x in step_bytes)
    # Every launch in the timed region is one of the attention call's kernels
    # (the host steps launch nothing), so the region's device time per step
    # is the call's average duration when the host keeps ahead of the GPU,
    # and an upper bound on it otherwise: this rank's roofline figure.
    call_ms = ms / args.steps
    attn_gbs = dram_rank / args.steps / (call_ms * 1e-3) / 1e9
    # A second, conservative reading after the timed region: single calls,
    # each between two events.  An event between two kernels ends their
    # programmatic overlap, so an isolated call is slower than one inside the
    # chain of steps.
    iso = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(10)]
    iso_bytes = [step(pair)[0] for pair in iso]
    torch.cuda.synchronize()
    iso_ms = float(np.mean([a.elapsed_time(z) for a, z in iso]))
    iso_gbs = float(np.mean(iso_bytes)) / (iso_ms * 1e-3) / 1e9
    peak, peak_kind = load_peaks()
    if cascade is not None:
        step_kernels = (("cascade_plan_kernel (with the table sync)" if runner.cascade_sync else
                         "seqtab_sync_kernel, cascade_plan_kernel")
                        + ", paged_attn_kernel (suffixes, fused append) beside cascade_prefix_kernel, combine_kernel")
    elif args.separate_append:
        step_kernels = "seqtab_sync_kernel, append_kernel, paged_attn_kernel, combine_kernel"
    elif multi:
        step_kernels = "paged_attn_kernel per batch (fused append, one chain), then combine_kernel per batch"
    elif fuse_sync:
        step_kernels = "paged_attn_kernel (fused append and table sync), combine_kernel"
    else:
        step_kernels = (("seqtab_sync_kernel, " if any(t is not None for t, _ in wl.tables()) else "")
                        + "paged_attn_kernel (fused append), combine_kernel")

    # end to end: each step's q / k / v come from pinned host memory and its
    # output goes back to pinned host memory.  The C-ABI calls get the host
    # buffers themselves: the kernels read the inputs and write the output
    # across the GPU's coherent host link (NVLink-C2C on GB300) inside the
    # step, so no copy-engine transfer splits the step's kernel chain.
    bufs = [buf for _, buf in wl.tables()]
    pinned = []
    for buf in bufs:
        pinned.append([torch.empty(buf.inputs.shape, dtype=torch.bfloat16).pin_memory().copy_(buf.inputs.cpu()),
                       torch.empty(buf.out.shape, dtype=torch.bfloat16).pin_memory()])
    h2d = sum(int(p[0].numel()) * 2 for p in pinned) + sum(b.rows * 4 for b in bufs)
    d2h = sum(int(p[1].numel()) * 2 for p in pinned)
    for buf, p in zip(bufs, pinned):
        buf.io(p[0], p[1])

    def e2e_step():
        return step()

    for i in range(3):
        e2e_step()
    torch.cuda.synchronize()
    e0 = torch.cuda.Event(enable_timing=True)
    e1 = torch.cuda.Event(enable_timing=True)
    e2e_bytes = 0
    e0.record(stream)
    for i in range(args.steps):
        e2e_bytes += e2e_step()[0]
    e1.record(stream)
    torch.cuda.synchronize()
    e2e_ms = e0.elapsed_time(e1)
    gc.enable()
    for buf in bufs:
        buf.io()
    ms, e2e_ms, tot = aggregate_ranks(dist, torch.device("cuda", local), ms, e2e_ms,
                                      {"dram": dram_rank, "logical": logical_rank, "tokens": wl.S * args.steps,
                                       "e2e": e2e_bytes})
    gbs = tot["dram"] / (ms * 1e-3) / 1e9
    tokens_per_s = tot["tokens"] / (ms * 1e-3)
    e2e_gbs = tot["e2e"] / (e2e_ms * 1e-3) / 1e9

    secondary = None
    if world == 1 and not args.no_secondary and args.workload == "llama8b":
        # the other workloads' steps, so that one run records all of them
        del bufs, pinned
        secondary = {}
        for name in ("chains", "coloc", "longctx"):
            secondary[name] = measure_secondary(name, args, K, W, DevicePool, DeviceSteps, stream, peak)

    cpu = None
    if rank == 0 and not args.no_cpu_baseline and args.workload == "llama8b":
        b = wl.b
        v, nst, el = oracle_baseline(b, args.cpu_budget)
        cpu = {"value": v, "unit": "GB/s", "cores": 1, "kind": "oracle",
               "sample": f"{nst} whole decode steps (append + attention over all {b.S} sequences) of the same "
                         f"workload, single-threaded C fp64, {el:.1f} s",
               "cpu_model": cpu_model(), "affinity_cores": len(all_cores) if all_cores else None}
        if all_cores and len(all_cores) > 1:
            vp, nsp, elp, T = oracle_baseline_parallel(b, args.cpu_budget, all_cores)
            cpu["all_cores"] = {"value": vp, "unit": "GB/s", "cores": T, "kind": "oracle",
                                "sample": f"{nsp} whole decode steps, the attention's sequences over {T} threads "
                                          f"(one per core; the append in place, on one), {elp:.1f} s"}

    traffic = None
    prof = os.path.join(ROOT, "profiles", "traffic.json")
    if args.workload == "llama8b" and os.path.exists(prof):
        try:
            with open(prof) as f:
                traffic = json.load(f).get("paged_attn_llama8b_bytes_per_launch")
        except Exception:
            traffic = None

    config = {"workload": wl.name, **wl.config, "num_splits": args.num_splits, "variant": args.variant,
              "pool": args.pool if args.workload == "llama8b" else "fixed",
              "append": "separate kernel" if args.separate_append else "fused into attention",
              "table_sync": ("carried by the decode launch when it fits" if fuse_sync else
                             "carried by the plan launch when it fits" if cascade_sync else "separate kernel"),
              "batches": "one paged_decode_attn_multi call" if multi else "one call per batch",
              "step_overlap": runner.step_overlap,
              "shared_prefix": ("attended once per KV head for all sharers (cascade)" if cascade is not None
                                else "streamed per sequence") if hasattr(wl, "prefix_plan") else None,
              "parallelism": f"replicas x{world}" if world > 1 else "single GPU"}
    line = {
        "metric": METRIC, "value": gbs, "unit": "GB/s", "n_gpus": world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": ms / args.steps, "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "bf16", "data": "synthetic", "config": config,
        "decode_tokens_per_s": tokens_per_s,
        "roofline": {"bound": "hbm", "achieved": attn_gbs, "peak": peak, "unit": "GB/s",
                     "frac": attn_gbs / peak, "traffic": traffic,
                     "kernel": step_kernels,
                     "peak_kind": peak_kind, "call_ms": call_ms, "timed_launches": runner.launches_per_step * args.steps
                     + extra_sync_launches,
                     "timing": "CUDA events at the ends of the timed region, whose launches are all the "
                               "attention call's kernels: region time / steps",
                     "isolated_call_ms": iso_ms, "isolated_frac": iso_gbs / peak},
        "step_frac_of_peak": gbs / world / peak,
        "e2e": {"value": e2e_gbs, "unit": "GB/s", "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h},
        "gpu_launches": runner.launches_per_step * args.steps + extra_sync_launches,
        "host_us_per_step": host_us,
        "host_cores": pinned_cores,
        "clocks": clk,
        "device_error": err,
        "cpu_baseline": cpu,
    }
    if secondary is not None:
        line["secondary_workloads"] = secondary
    if tot["logical"] != tot["dram"]:
        line["logical_gbs"] = tot["logical"] / (ms * 1e-3) / 1e9
    if rank == 0:
        print(json.dumps(line), flush=True)
    if dist:
        dist.barrier()
        dist.destroy_process_group()


if __name__ == "__main__":
    main()
