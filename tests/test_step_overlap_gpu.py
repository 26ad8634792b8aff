"""Step overlap (kv_set_attn_step_overlap): a decode kernel that starts while
the previous step's split-K combine on the same stream finishes must give
the bits of one that waits for it.

Two pools with the same contents and the same host sequence tables run the
config-2 batch (64 sequences, lognormal contexts, one appended token per
step) through paged_decode_attn_seqtab with the fused append, one with the
overlap on and one with it off: steps back to back on one stream (only the
final output and the pool are compared, since any copy between the steps
would separate them), steps with an output copy between them, steps with
the pool's error read between them (a library copy, which turns the
overlap off for the next call), and automatic and forced split counts;
also pinned host buffers (the benchmark's end-to-end form) and two batches
on two streams with their steps interleaved.  The final output is checked
against the fp64 oracle, every sequence.
"""
import numpy as np
import pytest

import oracle
from paper_2606_12950_gb300 import kvpool as K
from paper_2606_12950_gb300 import workloads as W
from tests import par_oracle

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

MAX_ABS = 1.5e-2
MEAN_ABS = 2e-3


@pytest.fixture(scope="module", autouse=True)
def _cuda():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")


def _side(b, overlap, steps, num_splits):
    from paper_2606_12950_gb300.runner import DevicePool, DeviceSteps

    pool = DevicePool(b.n_pages, b.page_elems * 2, b.bs, [(b.Hkv, b.d)], shuffle_seed=b.meta["seed"])
    pool.upload(b.pool)
    pool.set_step_overlap(overlap)
    t = K.SeqTab(pool.handle, 0, b.S, b.max_blocks)
    pre = b.meta["pre_lens"].astype(np.int64)
    for s in range(b.S):
        t.reserve(s, int(pre[s]) + steps + 8)
        t.set_len(s, int(pre[s]))
    buf = DeviceSteps(pool, 0, b.S, b.S, b.Hq, b.Hkv, b.d, b.max_blocks, b.scale, b.q, b.k_new, b.v_new,
                      num_splits)
    return pool, t, buf


def _run(side, steps, between):
    """`steps` steps on the current stream; between(i) runs after step i
    (None: nothing between the steps).  Returns the per-step output copies."""
    pool, t, buf = side
    outs = []
    for i in range(steps):
        t.advance()
        buf.sync_append_attend(t)
        if between == "copy":
            outs.append(buf.out.clone())
        elif between == "error":
            assert pool.error() == 0
    torch.cuda.synchronize()
    return outs


@pytest.mark.parametrize("between", [None, "copy", "error"])
@pytest.mark.parametrize("num_splits", [0, 48])
def test_step_overlap_gives_the_bits_of_waiting_steps(between, num_splits):
    steps = 10
    b = W.config2_llama8b(steps=steps + 8)
    on = _side(b, True, steps, num_splits)
    off = _side(b, False, steps, num_splits)
    outs_on = _run(on, steps, between)
    outs_off = _run(off, steps, between)
    for i, (x, y) in enumerate(zip(outs_on, outs_off)):
        assert torch.equal(x.view(torch.int16), y.view(torch.int16)), i
    (pool_on, t_on, buf_on), (pool_off, t_off, buf_off) = on, off
    assert torch.equal(buf_on.out.view(torch.int16), buf_off.out.view(torch.int16))
    assert torch.equal(buf_on.table, buf_off.table) and torch.equal(buf_on.lens, buf_off.lens)
    got_pool = pool_on.download()
    assert np.array_equal(got_pool, pool_off.download())
    assert pool_on.error() == 0 and pool_off.error() == 0
    if between is None and num_splits == 0:
        # the final step against the oracle: the pool as appended by every
        # step (the host table names the rows), every sequence
        table, lens = t_on.host()
        host_pool = b.pool.copy()
        for i in range(steps):
            # every step appends the same new rows at position n-1
            lens_i = b.meta["pre_lens"].astype(np.int32) + i + 1
            oracle.append(host_pool, b.n_pages, b.page_elems, b.bs, b.Hkv, b.d, b.k_new, b.v_new, table,
                          lens_i, inplace=True)
        assert np.array_equal(got_pool, host_pool)
        ref = par_oracle.paged_attention(host_pool, b.n_pages, b.page_elems, b.bs, b.Hkv, b.d, b.q, table,
                                         lens, b.scale)
        got = buf_on.out.float().cpu().numpy().astype(np.float64)
        err = np.abs(got - ref)
        assert np.isfinite(got).all() and err.max() <= MAX_ABS and err.mean() <= MEAN_ABS, (err.max(), err.mean())
    for pool, t, _ in (on, off):
        t.close()
        pool.close()


def test_step_overlap_with_host_buffers():
    """The end-to-end form the benchmark times: q, k_new, v_new and out in
    pinned host memory that the kernels read and write directly, steps back
    to back with the overlap on; the same bits as device buffers with the
    overlap off."""
    steps = 6
    b = W.config2_llama8b(steps=steps + 8)
    on = _side(b, True, steps, 0)
    off = _side(b, False, steps, 0)
    pool_on, _, buf_on = on
    hin = torch.empty(buf_on.inputs.shape, dtype=torch.bfloat16).pin_memory()
    hin.copy_(buf_on.inputs.view(torch.bfloat16).cpu())
    hout = torch.full(buf_on.out.shape, float("nan"), dtype=torch.bfloat16).pin_memory()
    buf_on.io(hin, hout)
    _run(on, steps, None)
    _run(off, steps, None)
    assert torch.equal(hout.view(torch.int16), off[2].out.cpu().view(torch.int16))
    assert np.array_equal(pool_on.download(), off[0].download())
    assert pool_on.error() == 0 and off[0].error() == 0
    for pool, t, _ in (on, off):
        t.close()
        pool.close()


def test_step_overlap_on_two_streams():
    """Two batches on two streams, their steps interleaved on the host with
    the overlap on: each stream's record of the library's last launch is its
    own, so each batch gives the bits it gives alone with the overlap off."""
    steps = 6
    b = W.config2_llama8b(steps=steps + 8)
    sides = [_side(b, True, steps, 0), _side(b, True, steps, 0)]
    streams = [torch.cuda.Stream(), torch.cuda.Stream()]
    torch.cuda.synchronize()
    for i in range(steps):
        for (pool, t, buf), st in zip(sides, streams):
            t.advance()
            buf.sync_append_attend(t, st)
    torch.cuda.synchronize()
    ref = _side(b, False, steps, 0)
    _run(ref, steps, None)
    for pool, t, buf in sides:
        assert torch.equal(buf.out.view(torch.int16), ref[2].out.view(torch.int16))
        assert np.array_equal(pool.download(), ref[0].download())
        assert pool.error() == 0
    for pool, t, _ in sides + [ref]:
        t.close()
        pool.close()
