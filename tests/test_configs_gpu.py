"""Full-size parity of the multi-agent, co-location and long-context
workloads (configs 3, 4, 5), through the C ABI, against the fp64 oracle.

The block tables come from the library's host sequence tables (host code,
not the CUDA path); the oracle mirrors every append on its own copy of the
pool.  Every sequence's output is compared with the oracle on every checked
step (the oracle spread over the host cores, ``par_oracle``), the pool
bit-exactly.  The full-size tests drive the entry points and launch
configuration the benchmark times for each workload: the cascade call with
the fused append and the table sync carried by its plan kernel (agent
chains), one
paged_decode_attn_multi call (co-location), paged_decode_attn_seqtab with
the fused sync and append (long context).
"""
import numpy as np
import pytest

import oracle
from tests import par_oracle
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


def _check(got, ref, what):
    err = np.abs(got - ref)
    assert np.isfinite(got).all(), what
    assert err.max() <= MAX_ABS and err.mean() <= MEAN_ABS, (what, err.max(), err.mean())


def _check_all(got, host_pool, n_pages, page_elems, bs, Hkv, d, q, table, lens, scale, what):
    """Every sequence of the batch against the oracle."""
    ref = par_oracle.paged_attention(host_pool, n_pages, page_elems, bs, Hkv, d, q, table, lens, scale)
    _check(got, ref, what)


def _run_chains(n_chains, steps, median, max_out, seed=1003, check_every=1, cascade=False,
                until_stage_end=False, sync_in_call=False, bits=None, pages_per_chain=150):
    """Agent chains driven as the benchmark drives them: the sequence table's
    sync, then the cascade call with the fused append (shared-prefix mode;
    with sync_in_call one paged_decode_attn_cascade_seqtab call, the sync
    carried by its plan kernel) or the append and attention calls.  Every
    chain is checked on every checked step.  With until_stage_end the run
    goes on (up to ``steps``) until two steps after the first stage
    boundary.  ``bits``, a list, receives every step's output bits, device
    lengths and table, and the run's sync-kernel launches after each step."""
    from paper_2606_12950_gb300.runner import DevicePool, DeviceSteps
    from paper_2606_12950_gb300.schedules import AgentChains

    d, Hq, Hkv, bs = 128, 32, 8, 16
    max_blocks = (W.PREFIX_TOKENS + 4 * max_out * 2) // bs + 8
    n_pages = 128 + n_chains * pages_per_chain + 64  # about twice the expected need
    page_elems = 2 * Hkv * bs * d
    host_pool = np.empty(n_pages * page_elems, np.uint16)
    W.bf16_normal_fill(host_pool, seed + 7919)
    pool = DevicePool(n_pages, page_elems * 2, bs, [(Hkv, d)], shuffle_seed=seed)
    pool.upload(host_pool)
    ch = AgentChains(pool.handle, 0, n_chains, max_blocks, bs, seed, median=median, max_out=max_out)
    q, kn, vn = W.step_rows(seed, 0, n_chains, Hq, Hkv, d)
    buf = DeviceSteps(pool, 0, n_chains + 1, n_chains, Hq, Hkv, d, max_blocks, d ** -0.5, q, kn, vn)
    plan = ch.prefix_plan() if cascade else None
    if cascade:
        buf.use_cascade()
    boundary_step = None
    checked = 0
    for step in range(steps):
        ch.step()
        q, kn, vn = W.step_rows(seed, step, n_chains, Hq, Hkv, d)
        buf.inputs.copy_(_dev_bits(np.concatenate([q.reshape(-1), kn.reshape(-1), vn.reshape(-1)])))
        if cascade and sync_in_call:
            buf.sync_cascade(ch.tab, plan)
        elif cascade:
            buf.sync(ch.tab)
            buf.cascade(plan)
        else:
            buf.sync(ch.tab)
            buf.append()
            buf.attend()
        torch.cuda.synchronize()
        got = buf.out.float().cpu().numpy().astype(np.float64)
        if bits is not None:
            bits.append((buf.out.view(torch.int16).cpu().numpy().copy(), buf.lens.cpu().numpy().copy(),
                         buf.table.cpu().numpy().copy(), ch.tab.counters()["sync_launches"]))
        table, lens = ch.tab.host()
        table, lens = table[:n_chains], lens[:n_chains]
        oracle.append(host_pool, n_pages, page_elems, bs, Hkv, d, kn, vn, table, lens, inplace=True)
        if boundary_step is None and ch.stage_ends > 0:
            boundary_step = step
        if step % check_every == 0 or step == steps - 1 or boundary_step is not None:
            _check_all(got, host_pool, n_pages, page_elems, bs, Hkv, d, q, table, lens, d ** -0.5,
                       f"chains step {step}")
            checked += 1
        if until_stage_end and boundary_step is not None and step >= boundary_step + 2:
            break
    assert np.array_equal(pool.download(), host_pool)
    assert pool.error() == 0
    stats = (ch.stage_ends, ch.chains_done, ch.tab.counters()["reservation_misses"], boundary_step, checked)
    ch.close()
    pool.close()
    return stats


def test_agent_chains_full_size():
    """256 concurrent chains, 2048-token shared prefix, stage outputs
    lognormal(300), reservations true x U[0.8, 1.5]; the prefix streamed per
    chain; every chain checked on 3 steps."""
    _run_chains(256, steps=3, median=300.0, max_out=4096)


def test_agent_chains_full_size_cascade_across_a_stage_boundary():
    """The same 256 chains through shared-prefix attention, as the benchmark
    runs them (one cascade call with the fused append, the table sync
    carried by its plan kernel): the
    2048-token prompt attended once per KV head for all chains, each chain's
    own context streamed and merged.  The run goes past the first stage
    boundary (a trim and a new stage's reservation; with this seed the
    first stage ends at step 24); every chain is checked on every fourth
    step and on every step from the boundary on."""
    ends, done, misses, boundary, checked = _run_chains(256, steps=64, median=300.0, max_out=4096,
                                                        check_every=4, cascade=True, until_stage_end=True,
                                                        sync_in_call=True)
    assert boundary is not None and ends >= 1 and checked >= 8


def test_table_sync_carried_by_the_plan_kernel_gives_the_separate_sync_bits():
    """paged_decode_attn_cascade_seqtab against kv_seqtab_sync followed by
    paged_decode_attn_cascade, on the same short-stage schedule (stage ends,
    trims, chain releases, new chains re-sharing the prefix): on every step
    the same output bits, device lengths and table; the first step (a table
    never written to the device) takes the separate sync, every later one
    launches no sync kernel; both runs match the oracle on every fourth
    step."""
    fused, separate = [], []
    _run_chains(48, steps=40, median=5.0, max_out=40, check_every=4, cascade=True, sync_in_call=True,
                bits=fused)
    _run_chains(48, steps=40, median=5.0, max_out=40, check_every=4, cascade=True, bits=separate)
    assert len(fused) == len(separate) == 40
    for i, (f, r) in enumerate(zip(fused, separate)):
        for a, b in zip(f[:3], r[:3]):
            assert np.array_equal(a, b), i
    assert fused[0][3] >= 1 and fused[-1][3] == fused[0][3]  # no sync kernel after the first step
    assert separate[-1][3] >= separate[0][3] + 39


def test_table_sync_too_large_for_the_plan_kernel_runs_first():
    """1500 chains: the plan (about 3000 words) and the table's 1501 lengths
    exceed the plan kernel's 4080-word block, so paged_decode_attn_cascade_seqtab
    runs the sync kernel first on every step; the bits still equal the
    separate sync followed by the cascade call, and the run matches the
    oracle on the first and last of six steps."""
    fused, separate = [], []
    _run_chains(1500, steps=6, median=5.0, max_out=40, check_every=5, cascade=True, sync_in_call=True,
                bits=fused, pages_per_chain=16)
    _run_chains(1500, steps=6, median=5.0, max_out=40, check_every=5, cascade=True, bits=separate,
                pages_per_chain=16)
    for i, (f, r) in enumerate(zip(fused, separate)):
        for a, b in zip(f[:3], r[:3]):
            assert np.array_equal(a, b), i
    assert fused[-1][3] >= fused[0][3] + 5  # a sync kernel on every step


def test_agent_chains_stage_turnover_cascade():
    ends, done, misses, _, _ = _run_chains(48, steps=40, median=5.0, max_out=40, check_every=4, cascade=True)
    assert ends > 48 and done > 0 and misses > 0


def test_agent_chains_stage_turnover():
    """Short stages so that stage ends, trims, chain releases and new chains
    (re-sharing the prefix) all happen within the run; every chain checked."""
    ends, done, misses, _, _ = _run_chains(48, steps=40, median=5.0, max_out=40, check_every=4)
    assert ends > 48 and done > 0 and misses > 0


def test_colocated_models_full_size():
    """Three layer shapes in one pool filled to 90% (MHA 32/32, GQA 32/8,
    GQA 40/8), 512 sequences, bounded-Pareto(1.5) lengths: one decode step
    per layout, separate append and attention calls; every sequence checked."""
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
    for li, (b, db) in enumerate(zip(batches, dbs)):
        oracle.append(host_pool, n_pages, page_elems, b.bs, b.Hkv, b.d, b.k_new, b.v_new, b.table, b.ctx_lens,
                      inplace=True)
    assert np.array_equal(pool.download(), host_pool)
    for li, (b, db) in enumerate(zip(batches, dbs)):
        _check_all(db.out_f64(), host_pool, n_pages, page_elems, b.bs, b.Hkv, b.d, b.q, b.table, b.ctx_lens,
                   b.scale, f"layout {li}")
    assert pool.error() == 0
    pool.close()


def test_colocated_models_in_one_multi_call():
    """The three co-located batches in one paged_decode_attn_multi call with
    the fused append, buffers held as the benchmark holds them (DeviceSteps,
    tables uploaded once): outputs and pool bit-identical to three
    paged_decode_attn_append calls, all 512 sequences against the oracle,
    the pool against the oracle's.  A batch with S = 0 in the list is
    skipped."""
    from paper_2606_12950_gb300 import kvpool as K
    from paper_2606_12950_gb300.runner import DeviceBatch, DevicePool, DeviceSteps

    batches, n_pages, page_elems = W.config4_colocation()
    pool_a = DevicePool(n_pages, page_elems * 2, 16, [(b.Hkv, b.d) for b in batches])
    pool_a.upload(batches[0].pool)
    dbs_a = [DeviceBatch(pool_a, li, b) for li, b in enumerate(batches)]
    for db in dbs_a:
        db.append_attend()
    pool_b = DevicePool(n_pages, page_elems * 2, 16, [(b.Hkv, b.d) for b in batches])
    pool_b.upload(batches[0].pool)
    bufs = []
    for li, b in enumerate(batches):
        buf = DeviceSteps(pool_b, li, b.S, b.S, b.Hq, b.Hkv, b.d, b.max_blocks, b.scale, b.q, b.k_new, b.v_new)
        K.kv_block_table_upload(pool_b.handle, li, b.table, b.ctx_lens, buf.table, buf.lens)
        bufs.append(buf)
    entries = [buf.batch() for buf in bufs]
    empty = dict(entries[1], S=0)
    K.paged_decode_attn_multi(pool_b.handle, [entries[0], empty, entries[1], entries[2]])
    torch.cuda.synchronize()
    got_pool = pool_b.download()
    assert np.array_equal(pool_a.download(), got_pool)
    for li in range(3):
        assert np.array_equal(dbs_a[li].out_bits(),
                              bufs[li].out.view(torch.int16).cpu().numpy().view(np.uint16)), f"layout {li}"
    host_pool = batches[0].pool.copy()
    for b in batches:
        oracle.append(host_pool, n_pages, page_elems, b.bs, b.Hkv, b.d, b.k_new, b.v_new, b.table, b.ctx_lens,
                      inplace=True)
    assert np.array_equal(got_pool, host_pool)
    for li, (b, buf) in enumerate(zip(batches, bufs)):
        got = buf.out.float().cpu().numpy().astype(np.float64)
        _check_all(got, host_pool, n_pages, page_elems, b.bs, b.Hkv, b.d, b.q, b.table, b.ctx_lens, b.scale,
                   f"layout {li}")
    assert pool_a.error() == 0 and pool_b.error() == 0
    pool_a.close()
    pool_b.close()


def test_long_context_stress_full_size():
    """1024 sequences, bounded-Pareto(1.2) contexts on [256, 131072], bs=32,
    driven as the benchmark drives it: paged_decode_attn_seqtab with the
    fused append (its 1024 lengths do not fit the decode kernel's parameter
    block, so the sync kernel runs first), the workspace sized for automatic
    splits.  Ten steps: sequences finish, their blocks go back to the free
    lists and new sequences are admitted into them (over 150 by step 9 with
    this seed).  Every sequence checked on every step, the pool at the end."""
    from paper_2606_12950_gb300.runner import DevicePool, DeviceSteps
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
    q, kn, vn = W.step_rows(seed, 0, S, Hq, Hkv, d)
    buf = DeviceSteps(pool, 0, S, S, Hq, Hkv, d, max_blocks, d ** -0.5, q, kn, vn)
    syncs0 = lc.tab.counters()["sync_launches"]
    for step in range(10):
        lc.step()
        q, kn, vn = W.step_rows(seed, step, S, Hq, Hkv, d)
        buf.inputs.copy_(_dev_bits(np.concatenate([q.reshape(-1), kn.reshape(-1), vn.reshape(-1)])))
        buf.sync_append_attend(lc.tab)
        torch.cuda.synchronize()
        got = buf.out.float().cpu().numpy().astype(np.float64)
        table, lens = lc.tab.host()
        live = lens > 0
        oracle.append(host_pool, n_pages, page_elems, bs, Hkv, d, kn, vn, table, lens, inplace=True)
        ref = par_oracle.paged_attention(host_pool, n_pages, page_elems, bs, Hkv, d, q, table, lens, d ** -0.5)
        _check(got[live], ref[live], f"long step {step}")
        assert not got[~live].any()  # an empty slot's output is zeros
    assert lc.released > 100 and lc.admitted > S + 100
    assert lc.tab.counters()["sync_launches"] - syncs0 >= 10  # every step's sync ran as its own kernel
    assert np.array_equal(pool.download(), host_pool)
    assert pool.error() == 0
    lc.close()
    pool.close()
