"""Step overlap of shared-prefix calls (kv_set_attn_step_overlap): a
paged_decode_attn_cascade_seqtab call whose stream last received the
combine of the previous shared-prefix call on the same workspace starts
while that combine finishes.  Its plan kernel writes the plan, the skips
(into the skip array the combine does not read) and the table sync at once
and raises its first flag; the prefix kernel releases the decode kernel
before its own wait; the decode kernel reads after the first flag and
writes its output and partials after the second, which the plan kernel
raises once the combine has completed.  Results must be the bits of steps
that wait.

Two pools with the same contents run the same host schedule of agent
chains (one 2048-token prompt shared by reference; short stages, so that
stage ends, trims, releases and new chains re-sharing the prompt reach the
plan kernel as table changes), one with the overlap on and one with it off:
- steps back to back on one stream (the final output, lengths, table and
  pool compared: a copy between the steps would separate them);
- the full-size agent chains (256 chains), as the benchmark runs them;
- 600 chains, whose plan and sync take the plan kernel's larger parameter
  block;
- an output copy and new inputs between steps (every step compared);
- the pool's error word read between some steps (a library copy: the next
  call does not overlap);
- two batches with their own workspaces interleaved on one stream (no
  call follows a combine on its own workspace, so none overlaps).
The pool's counter shows which calls overlapped; outputs are checked
against the fp64 oracle on every sequence, the pool bit-exactly.
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
D, HQ, HKV, BS = 128, 32, 8, 16


@pytest.fixture(scope="module", autouse=True)
def _cuda():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")


def _dev_bits(a):
    return torch.from_numpy(np.ascontiguousarray(a).view(np.int16)).cuda().view(torch.bfloat16)


class Side:
    """A pool, its agent chains and their decode buffers; the host pool
    mirrors every append for the oracle."""

    def __init__(self, n_chains, median, max_out, overlap, seed=1003, pages_per_chain=150):
        from paper_2606_12950_gb300.runner import DevicePool, DeviceSteps
        from paper_2606_12950_gb300.schedules import AgentChains

        self.n, self.seed = n_chains, seed
        self.max_blocks = (W.PREFIX_TOKENS + 4 * max_out * 2) // BS + 8
        self.n_pages = 128 + n_chains * pages_per_chain + 64
        self.page_elems = 2 * HKV * BS * D
        self.host_pool = np.empty(self.n_pages * self.page_elems, np.uint16)
        W.bf16_normal_fill(self.host_pool, seed + 7919)
        self.pool = DevicePool(self.n_pages, self.page_elems * 2, BS, [(HKV, D)], shuffle_seed=seed)
        self.pool.upload(self.host_pool)
        self.pool.set_step_overlap(overlap)
        self.ch = AgentChains(self.pool.handle, 0, n_chains, self.max_blocks, BS, seed, median=median,
                              max_out=max_out)
        self.q, self.kn, self.vn = W.step_rows(seed, 0, n_chains, HQ, HKV, D)
        self.buf = DeviceSteps(self.pool, 0, n_chains + 1, n_chains, HQ, HKV, D, self.max_blocks, D ** -0.5,
                               self.q, self.kn, self.vn)
        self.buf.use_cascade()
        self.plan = self.ch.prefix_plan()
        # a library copy on the stream: no earlier combine counts for the first call
        assert self.pool.error() == 0
        self.overlapped0 = self.overlapped()
        self.separate = []  # per step: the call ran the table sync kernel first
        self.pending = []   # steps whose appends the host pool does not hold yet

    def overlapped(self):
        return K.kv_pool_stats(self.pool.handle)["attn_calls_overlapped"]

    def new_inputs(self, step):
        self.q, self.kn, self.vn = W.step_rows(self.seed, step, self.n, HQ, HKV, D)
        self.buf.inputs.copy_(_dev_bits(np.concatenate([self.q.reshape(-1), self.kn.reshape(-1),
                                                        self.vn.reshape(-1)])))

    def step(self, stream=None):
        """host schedule, then the call; returns this step's host table and
        lengths (the first n rows).  The host pool's copy of the step's
        append waits for mirror(), so that steps reach the GPU back to back."""
        self.ch.step()
        before = self.sync_launches()
        self.buf.sync_cascade(self.ch.tab, self.plan, stream=stream)
        self.separate.append(self.sync_launches() > before)
        table, lens = self.ch.tab.host()
        table, lens = table[:self.n].copy(), lens[:self.n].copy()
        self.pending.append((self.kn, self.vn, table, lens))
        return table, lens

    def mirror(self):
        for kn, vn, table, lens in self.pending:
            oracle.append(self.host_pool, self.n_pages, self.page_elems, BS, HKV, D, kn, vn, table, lens,
                          inplace=True)
        self.pending = []

    def check(self, table, lens, what):
        self.mirror()
        got = self.buf.out.float().cpu().numpy().astype(np.float64)
        ref = par_oracle.paged_attention(self.host_pool, self.n_pages, self.page_elems, BS, HKV, D, self.q, table,
                                         lens, D ** -0.5)
        err = np.abs(got - ref)
        assert np.isfinite(got).all(), what
        assert err.max() <= MAX_ABS and err.mean() <= MEAN_ABS, (what, err.max(), err.mean())

    def bits(self):
        return (self.buf.out.view(torch.int16).cpu().numpy().copy(), self.buf.lens.cpu().numpy().copy(),
                self.buf.table.cpu().numpy().copy())

    def sync_launches(self):
        return self.ch.tab.counters()["sync_launches"]

    def expected_overlaps(self):
        """calls after the first whose stream last received this workspace's
        combine: those that did not run the separate table sync first"""
        return sum(1 for sep in self.separate[1:] if not sep)

    def close(self):
        assert self.pool.error() == 0
        self.ch.close()
        self.pool.close()


def _equal(a, b, what):
    for x, y in zip(a, b):
        assert np.array_equal(x, y), what


def _back_to_back(n_chains, steps, median, max_out, pages_per_chain=150):
    on = Side(n_chains, median, max_out, True, pages_per_chain=pages_per_chain)
    off = Side(n_chains, median, max_out, False, pages_per_chain=pages_per_chain)
    for side in (on, off):
        for _ in range(steps):
            table, lens = side.step()
        torch.cuda.synchronize()
        side.mirror()
        side.final = (table, lens)
    _equal(on.bits(), off.bits(), "final output, lengths and table")
    assert np.array_equal(on.pool.download(), off.pool.download())
    assert np.array_equal(on.pool.download(), on.host_pool)
    on.check(*on.final, "final step, overlap on")
    # every call after the first overlapped, except those that ran the
    # separate table sync first (a library launch between the calls)
    assert on.separate[0] and on.expected_overlaps() >= steps // 2
    assert on.overlapped() - on.overlapped0 == on.expected_overlaps()
    assert off.overlapped() == off.overlapped0
    stats = (on.ch.stage_ends, on.ch.chains_done)
    on.close()
    off.close()
    return stats


def test_cascade_overlap_back_to_back_with_stage_turnover():
    """48 chains with short stages, 40 steps back to back on one stream."""
    ends, done = _back_to_back(48, steps=40, median=5.0, max_out=40)
    assert ends > 48 and done > 0


def test_cascade_overlap_full_size_agent_chains():
    """256 chains, stage outputs lognormal(300): 12 steps back to back."""
    _back_to_back(256, steps=12, median=300.0, max_out=4096)


def test_cascade_overlap_with_a_larger_plan():
    """600 chains: the plan (about 1200 words) and the sync take the plan
    kernel's 8 KB parameter block; 10 steps back to back."""
    _back_to_back(600, steps=10, median=5.0, max_out=40, pages_per_chain=16)


def test_cascade_overlap_with_copies_between_steps():
    """New inputs before and an output copy after every step (copies of
    others, which the library does not see: the next call still takes the
    overlapped path, and the copies order it after the combine); every
    step's bits compared, the oracle on every fourth step."""
    steps = 24
    on = Side(48, 5.0, 40, True)
    off = Side(48, 5.0, 40, False)
    res = {}
    for name, side in (("on", on), ("off", off)):
        out = []
        for step in range(steps):
            side.new_inputs(step)
            table, lens = side.step()
            out.append(side.bits())
            if step % 4 == 3:
                side.check(table, lens, f"{name} step {step}")
        res[name] = out
    for i, (x, y) in enumerate(zip(res["on"], res["off"])):
        _equal(x, y, f"step {i}")
    assert on.overlapped() - on.overlapped0 == on.expected_overlaps() >= steps // 2
    on.mirror()
    assert np.array_equal(on.pool.download(), on.host_pool)
    on.close()
    off.close()


def test_cascade_overlap_off_after_a_library_copy():
    """The pool's error word read (a copy and a clear by the library) after
    every third step: the call after it waits for the combine instead of
    overlapping it; the bits still match the overlap off, and the final
    output matches the oracle."""
    steps = 15
    on = Side(48, 5.0, 40, True)
    off = Side(48, 5.0, 40, False)
    for side in (on, off):
        after_copy = []
        for i in range(steps):
            after_copy.append(i > 0 and (i - 1) % 3 == 2)
            table, lens = side.step()
            if i % 3 == 2:
                assert side.pool.error() == 0
        torch.cuda.synchronize()
        side.final = (table, lens)
    _equal(on.bits(), off.bits(), "final output, lengths and table")
    expected = sum(1 for i in range(1, steps) if not on.separate[i] and not after_copy[i])
    assert expected >= steps // 2
    assert on.overlapped() - on.overlapped0 == expected
    on.check(*on.final, "final step, overlap on")
    on.mirror()
    assert np.array_equal(on.pool.download(), on.host_pool)
    on.close()
    off.close()


def test_cascade_calls_on_two_workspaces_do_not_overlap():
    """Two batches (their own pools, tables and workspaces) with their steps
    interleaved on one stream: every call follows the other batch's
    combine, so none overlaps; both match the oracle at the end."""
    a = Side(32, 5.0, 40, True, seed=1011)
    b = Side(32, 5.0, 40, True, seed=1013)
    s = torch.cuda.Stream()
    with torch.cuda.stream(s):
        for _ in range(10):
            fa = a.step(stream=s.cuda_stream)
            fb = b.step(stream=s.cuda_stream)
    s.synchronize()
    assert a.overlapped() == a.overlapped0 and b.overlapped() == b.overlapped0
    a.check(*fa, "batch a")
    b.check(*fb, "batch b")
    a.close()
    b.close()
