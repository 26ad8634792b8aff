"""The benchmark's multi-rank path on the CPU: two gloo ranks, each a
replica with its own work, reduce to the whole-job figures (the slowest
rank's time, the sum of the units), and the reference arm prints on rank 0
only."""
import json
import os
import socket
import subprocess
import sys

import numpy as np
import pytest

torch = pytest.importorskip("torch")
ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank(rank, world, port, out):
    import torch.distributed as dist

    sys.path.insert(0, ROOT)
    import bench

    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    dist.init_process_group("gloo", rank=rank, world_size=world)
    # rank r: 10 + r ms, bytes 100 * (r + 1), tokens 64 each
    got = bench.aggregate_ranks(dist, torch.device("cpu"), 10.0 + rank, 20.0 - rank,
                                {"dram": 100.0 * (rank + 1), "tokens": 64.0})
    with open(os.path.join(out, f"rank{rank}.json"), "w") as f:
        json.dump(got, f)
    dist.barrier()
    dist.destroy_process_group()


def test_aggregate_over_two_gloo_ranks(tmp_path):
    import torch.multiprocessing as mp

    port = _free_port()
    mp.start_processes(_rank, args=(2, port, str(tmp_path)), nprocs=2, join=True, start_method="spawn")
    for r in range(2):
        ms, e2e_ms, units = json.load(open(tmp_path / f"rank{r}.json"))
        assert ms == 11.0 and e2e_ms == 20.0  # the slowest rank's times
        assert units == {"dram": 300.0, "tokens": 128.0}  # every rank's units


def test_single_process_passes_through():
    sys.path.insert(0, ROOT)
    import bench

    assert bench.aggregate_ranks(None, None, 3.0, 4.0, {"a": 5}) == (3.0, 4.0, {"a": 5})


def test_reference_arm_prints_on_rank0_only():
    """Under torchrun only rank 0 runs and prints the oracle's line; rank 1
    exits 0 without work (here: two ranks launched by hand, no rendezvous
    needed because the reference arm makes none)."""
    env = dict(os.environ, WORLD_SIZE="2", RANK="1", LOCAL_RANK="1")
    r1 = subprocess.run([sys.executable, os.path.join(ROOT, "bench.py"), "--impl", "reference", "--steps", "1",
                         "--warmup", "0", "--gpus", "2"], env=env, capture_output=True, text=True, timeout=300)
    assert r1.returncode == 0 and r1.stdout.strip() == ""
    env.update(RANK="0", LOCAL_RANK="0")
    r0 = subprocess.run([sys.executable, os.path.join(ROOT, "bench.py"), "--impl", "reference", "--steps", "1",
                         "--warmup", "0", "--gpus", "2"], env=env, capture_output=True, text=True, timeout=600)
    assert r0.returncode == 0, r0.stderr[-2000:]
    lines = [l for l in r0.stdout.splitlines() if l.strip()]
    assert len(lines) == 1
    line = json.loads(lines[0])
    assert line["impl"] == "reference" and line["n_gpus"] == 2 and line["value"] > 0
    assert line["e2e"]["h2d_bytes_per_step"] == 0 and line["cpu_baseline"]["kind"] == "oracle"


def test_threaded_oracle_baseline_covers_every_sequence_once():
    """The all-cores oracle timing computes the same attention as one
    oracle call: the per-thread sequence subsets, merged, give the single
    call's output exactly, and the timing helper runs on a small batch."""
    sys.path.insert(0, ROOT)
    import numpy as np

    import bench
    import oracle
    from paper_2606_12950_gb300 import workloads as W

    b = W.make_batch(31, [5, 40, 17, 1, 64, 33, 9], Hq=4, Hkv=2, d=16, bs=4, extra_blocks=8)
    full = oracle.paged_attention(b.pool, b.n_pages, b.page_elems, b.bs, b.Hkv, b.d, b.q, b.table,
                                  b.ctx_lens, b.scale)
    T = 3
    order = np.argsort(-b.ctx_lens.astype(np.int64), kind="stable")
    merged = np.full_like(full, np.nan)
    for i in range(T):
        ids = order[i::T].astype(np.int32)
        part = oracle.paged_attention(b.pool, b.n_pages, b.page_elems, b.bs, b.Hkv, b.d, b.q, b.table,
                                      b.ctx_lens, b.scale, seq_ids=ids)
        assert np.isnan(part[np.setdiff1d(np.arange(b.S), ids)]).all()
        merged[ids] = part[ids]
    assert np.array_equal(merged, full)
    b.meta["seed"] = 31
    cores = set(sorted(os.sched_getaffinity(0))[:2])
    before = os.sched_getaffinity(0)
    gbs, steps, el, threads = bench.oracle_baseline_parallel(b, 0.0, cores)
    assert steps == 1 and gbs > 0 and threads == len(cores)
    assert os.sched_getaffinity(0) == before  # the caller's affinity is restored


def test_oracle_baselines_run_past_the_table_headroom():
    """Both oracle timings run more steps than the batch's table holds: the
    steps go in laps from the step-0 state, so no append leaves the
    reserved blocks (the fixed table holds 3 more appends here), and every
    lap's lengths are the step-0 lengths plus the lap's step index."""
    sys.path.insert(0, ROOT)
    import bench
    from paper_2606_12950_gb300 import workloads as W

    pre = [5, 40, 17, 1, 64, 33, 9]
    b = W.make_batch(37, pre, Hq=4, Hkv=2, d=16, bs=4, extra_blocks=8,
                     table_tokens=[p + 3 for p in pre])
    b.meta["seed"] = 37
    lap = bench.oracle_lap_steps(b)
    cap = (b.table >= 0).sum(axis=1) * b.bs
    assert lap == int((cap - b.ctx_lens).min()) + 1 and 1 <= lap <= 4
    gbs, steps, el = bench.oracle_baseline(b, 1e9, max_steps=5 * lap + 2)
    assert steps == 5 * lap + 2 and gbs > 0
    cores = set(sorted(os.sched_getaffinity(0))[:2])
    gbs, steps, el, threads = bench.oracle_baseline_parallel(b, 1e9, cores, max_steps=5 * lap + 2)
    assert steps == 5 * lap + 2 and gbs > 0 and threads == len(cores)


def test_oracle_baseline_on_the_benchmark_batch_at_the_driver_step_counts():
    """The benchmark's own batch at 20 steps + 5 warm-up: the oracle's
    laps fit its table however many steps the time budget allows."""
    sys.path.insert(0, ROOT)
    import bench
    from paper_2606_12950_gb300 import workloads as W

    b = W.config2_llama8b(steps=max(100, 2 * (5 + 20) + 8), fill_pool=False)
    lap = bench.oracle_lap_steps(b)
    cap = (b.table >= 0).sum(axis=1) * b.bs
    for i in range(lap):  # every appended position of a lap is inside its row's blocks
        assert np.all(b.ctx_lens + i - 1 < cap)
    assert np.any(b.ctx_lens + lap - 1 >= cap)
