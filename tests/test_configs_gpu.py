"""Full-size parity of the multi-agent, co-location and long-context
workloads (configs 3, 4, 5), through the C ABI, against the fp64 oracle.

The block tables come from the library's host sequence tables (host code,
not the CUDA path); the oracle mirrors every append on its own copy of the
pool.  Outputs are compared on sampled sequences (always including the
longest), the pool bit-exactly.
"""
import numpy as np
import pytest

import oracle
from paper_2606_12950_gb300 import kvpool as K
from paper_2606_12950_gb300 import workloads as W

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

MAX_ABS = 1.5e-2
MEAN_ABS = 2e-3


@pytest.fixture(scope="module", autouse=True)
def _cuda():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")


def _dev_bits(a):
    return torch.from_numpy(np.ascontiguousarray(a).view(np.int16)).cuda().view(torch.bfloat16)


class Runner:
    """Device buffers for one layout's decode batch driven by a sequence table."""

    def __init__(self, pool, layout, rows, max_blocks, Hq, Hkv, d, seed, scale):
        self.pool, self.layout = pool, layout
        self.rows, self.max_blocks, self.Hq, self.Hkv, self.d = rows, max_blocks, Hq, Hkv, d
        self.seed, self.scale = seed, scale
        self.table = torch.full((rows, max_blocks), -1, dtype=torch.int32, device="cuda")
        self.lens = torch.zeros(rows, dtype=torch.int32, device="cuda")

    def step(self, tab, S, step, plan=None):
        q, kn, vn = W.step_rows(self.seed, step, S, self.Hq, self.Hkv, self.d)
        qd, kd, vd = _dev_bits(q), _dev_bits(kn), _dev_bits(vn)
        out = torch.empty_like(qd)
        tab.sync(self.table, self.lens)
        if plan is not None:  # shared-prefix attention with the fused append
            nbytes = K.kv_cascade_workspace_bytes(self.pool.handle, self.layout, S, self.Hq, self.max_blocks)
            ws = torch.empty(nbytes, dtype=torch.uint8, device="cuda")
            K.paged_decode_attn_cascade(self.pool.handle, self.layout, qd, kd, vd, out, self.table, self.lens,
                                        self.max_blocks, S, self.Hq, self.scale, plan, ws, nbytes)
            torch.cuda.synchronize()
            return q, kn, vn, out.float().cpu().numpy().astype(np.float64)
        K.kv_append(self.pool.handle, self.layout, kd, vd, self.table, self.lens, self.max_blocks, S)
        nbytes = K.kv_workspace_bytes(self.pool.handle, self.layout, S, self.Hq, self.max_blocks)
        ws = torch.empty(nbytes, dtype=torch.uint8, device="cuda")
        K.paged_decode_attn(self.pool.handle, self.layout, qd, out, self.table, self.lens, self.max_blocks, S,
                            self.Hq, self.scale, 0, ws, nbytes)
        torch.cuda.synchronize()
        return q, kn, vn, out.float().cpu().numpy().astype(np.float64)


def _check(got, ref, what):
    err = np.abs(got - ref)
    assert np.isfinite(got).all(), what
    assert err.max() <= MAX_ABS and err.mean() <= MEAN_ABS, (what, err.max(), err.mean())


def _sample(rng, lens, k):
    order = np.argsort(lens)
    pick = set(int(x) for x in rng.choice(len(lens), size=min(k, len(lens)), replace=False))
    pick.add(int(order[-1]))
    return np.array(sorted(pick), np.int32)


def _run_chains(n_chains, steps, median, max_out, sample, seed=1003, check_every=1, cascade=False):
    from paper_2606_12950_gb300.runner import DevicePool
    from paper_2606_12950_gb300.schedules import AgentChains

    d, Hq, Hkv, bs = 128, 32, 8, 16
    max_blocks = (W.PREFIX_TOKENS + 4 * max_out * 2) // bs + 8
    n_pages = 128 + n_chains * 150 + 64  # about twice the expected need
    page_elems = 2 * Hkv * bs * d
    host_pool = np.empty(n_pages * page_elems, np.uint16)
    W.bf16_normal_fill(host_pool, seed + 7919)
    pool = DevicePool(n_pages, page_elems * 2, bs, [(Hkv, d)], shuffle_seed=seed)
    pool.upload(host_pool)
    ch = AgentChains(pool.handle, 0, n_chains, max_blocks, bs, seed, median=median, max_out=max_out)
    run = Runner(pool, 0, n_chains + 1, max_blocks, Hq, Hkv, d, seed, d ** -0.5)
    rng = np.random.default_rng(seed + 5)
    for step in range(steps):
        ch.step()
        q, kn, vn, got = run.step(ch.tab, n_chains, step, plan=ch.prefix_plan() if cascade else None)
        table, lens = ch.tab.host()
        table, lens = table[:n_chains], lens[:n_chains]
        oracle.append(host_pool, n_pages, page_elems, bs, Hkv, d, kn, vn, table, lens, inplace=True)
        if step % check_every == 0 or step == steps - 1:
            ids = _sample(rng, lens, sample) if sample else np.arange(n_chains, dtype=np.int32)
            ref = oracle.paged_attention(host_pool, n_pages, page_elems, bs, Hkv, d, q, table, lens, d ** -0.5,
                                         seq_ids=ids)
            _check(got[ids], ref[ids], f"chains step {step}")
    assert np.array_equal(pool.download(), host_pool)
    assert pool.error() == 0
    stats = (ch.stage_ends, ch.chains_done, ch.tab.counters()["reservation_misses"])
    ch.close()
    pool.close()
    return stats


def test_agent_chains_full_size():
    """256 concurrent chains, 2048-token shared prefix, stage outputs
    lognormal(300), reservations true x U[0.8, 1.5]."""
    _run_chains(256, steps=3, median=300.0, max_out=4096, sample=16)


def test_agent_chains_full_size_cascade():
    """The same 256 chains through shared-prefix attention: the 2048-token
    prompt is attended once per KV head for all chains, each chain's own
    context streamed and merged."""
    _run_chains(256, steps=3, median=300.0, max_out=4096, sample=16, cascade=True)


def test_agent_chains_stage_turnover_cascade():
    ends, done, misses = _run_chains(48, steps=40, median=5.0, max_out=40, sample=0, check_every=4, cascade=True)
    assert ends > 48 and done > 0 and misses > 0


def test_agent_chains_stage_turnover():
    """Short stages so that stage ends, trims, chain releases and new chains
    (re-sharing the prefix) all happen within the run; every chain checked."""
    ends, done, misses = _run_chains(48, steps=40, median=5.0, max_out=40, sample=0, check_every=4)
    assert ends > 48 and done > 0 and misses > 0


def test_colocated_models_full_size():
    """Three layer shapes in one pool filled to 90% (MHA 32/32, GQA 32/8,
    GQA 40/8), 512 sequences, bounded-Pareto(1.5) lengths: one decode step
    per layout."""
    from paper_2606_12950_gb300.runner import DeviceBatch, DevicePool

    batches, n_pages, page_elems = W.config4_colocation()
    pool = DevicePool(n_pages, page_elems * 2, 16, [(b.Hkv, b.d) for b in batches])
    pool.upload(batches[0].pool)
    host_pool = batches[0].pool.copy()
    dbs = [DeviceBatch(pool, li, b) for li, b in enumerate(batches)]
    for db in dbs:
        db.append()
    for db in dbs:
        db.attend()
    torch.cuda.synchronize()
    rng = np.random.default_rng(11)
    for li, (b, db) in enumerate(zip(batches, dbs)):
        oracle.append(host_pool, n_pages, page_elems, b.bs, b.Hkv, b.d, b.k_new, b.v_new, b.table, b.ctx_lens,
                      inplace=True)
    assert np.array_equal(pool.download(), host_pool)
    for li, (b, db) in enumerate(zip(batches, dbs)):
        ids = _sample(rng, b.ctx_lens, 12)
        ref = oracle.paged_attention(host_pool, n_pages, page_elems, b.bs, b.Hkv, b.d, b.q, b.table, b.ctx_lens,
                                     b.scale, seq_ids=ids)
        _check(db.out_f64()[ids], ref[ids], f"layout {li}")
    assert pool.error() == 0
    pool.close()


def test_colocated_models_in_one_multi_call():
    """The three co-located batches in one paged_decode_attn_multi call (the
    decode kernels chained, then the combines), with the fused append:
    outputs and pool bit-identical to three paged_decode_attn_append calls,
    and the oracle's values on sampled sequences.  A batch with S = 0 in the
    list is skipped."""
    from paper_2606_12950_gb300 import kvpool as K
    from paper_2606_12950_gb300.runner import DeviceBatch, DevicePool

    batches, n_pages, page_elems = W.config4_colocation()
    sides = []
    for _ in range(2):
        pool = DevicePool(n_pages, page_elems * 2, 16, [(b.Hkv, b.d) for b in batches])
        pool.upload(batches[0].pool)
        sides.append((pool, [DeviceBatch(pool, li, b) for li, b in enumerate(batches)]))
    pool_a, dbs_a = sides[0]
    for db in dbs_a:
        db.append_attend()
    pool_b, dbs_b = sides[1]
    entries = [db.batch() for db in dbs_b]
    empty = dict(entries[1], S=0)
    K.paged_decode_attn_multi(pool_b.handle, [entries[0], empty, entries[1], entries[2]])
    torch.cuda.synchronize()
    got_pool = pool_b.download()
    assert np.array_equal(pool_a.download(), got_pool)
    for li in range(3):
        assert np.array_equal(dbs_a[li].out_bits(), dbs_b[li].out_bits()), f"layout {li}"
    host_pool = batches[0].pool.copy()
    for b in batches:
        oracle.append(host_pool, n_pages, page_elems, b.bs, b.Hkv, b.d, b.k_new, b.v_new, b.table, b.ctx_lens,
                      inplace=True)
    assert np.array_equal(got_pool, host_pool)
    rng = np.random.default_rng(12)
    for li, (b, db) in enumerate(zip(batches, dbs_b)):
        ids = _sample(rng, b.ctx_lens, 8)
        ref = oracle.paged_attention(host_pool, n_pages, page_elems, b.bs, b.Hkv, b.d, b.q, b.table, b.ctx_lens,
                                     b.scale, seq_ids=ids)
        _check(db.out_f64()[ids], ref[ids], f"layout {li}")
    assert pool_a.error() == 0 and pool_b.error() == 0
    for pool, _ in sides:
        pool.close()


def test_long_context_stress_full_size():
    """1024 sequences, bounded-Pareto(1.2) contexts on [256, 131072], bs=32:
    steps with appends, sequences finishing, blocks freed and reused by new
    sequences."""
    from paper_2606_12950_gb300.runner import DevicePool
    from paper_2606_12950_gb300.schedules import LongContextStress

    seed, S, d, Hq, Hkv, bs = 1005, 1024, 128, 32, 8, 32
    max_blocks = (131072 + 64) // bs + 2
    est = int(W.config5_lengths(np.random.default_rng(seed), S).sum())
    n_pages = int(1.4 * est / bs) + 4096
    page_elems = 2 * Hkv * bs * d
    host_pool = np.empty(n_pages * page_elems, np.uint16)
    W.bf16_normal_fill(host_pool, seed + 7919)
    pool = DevicePool(n_pages, page_elems * 2, bs, [(Hkv, d)], shuffle_seed=seed)
    pool.upload(host_pool)
    lc = LongContextStress(pool.handle, 0, S, max_blocks, seed)
    run = Runner(pool, 0, S, max_blocks, Hq, Hkv, d, seed, d ** -0.5)
    rng = np.random.default_rng(seed + 5)
    for step in range(4):
        lc.step()
        q, kn, vn, got = run.step(lc.tab, S, step)
        table, lens = lc.tab.host()
        oracle.append(host_pool, n_pages, page_elems, bs, Hkv, d, kn, vn, table, lens, inplace=True)
        ids = _sample(rng, lens, 8)
        ref = oracle.paged_attention(host_pool, n_pages, page_elems, bs, Hkv, d, q, table, lens, d ** -0.5,
                                     seq_ids=ids)
        _check(got[ids], ref[ids], f"long step {step}")
    assert lc.released > 0 and lc.admitted > S
    assert np.array_equal(pool.download(), host_pool)
    assert pool.error() == 0
    lc.close()
    pool.close()
