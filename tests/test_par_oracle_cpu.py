"""The threaded oracle helper the full-size parity tests use gives the
single oracle call's result bit for bit, for the whole batch and for a
subset of it, at any thread count; and the oracle's own subset option
computes exactly the rows it is asked for."""
import numpy as np

import oracle
from paper_2606_12950_gb300 import workloads as W
from tests import par_oracle


def _batch():
    return W.make_batch(41, [5, 40, 17, 0, 64, 33, 9, 120, 1], Hq=6, Hkv=2, d=16, bs=4, extra_blocks=8)


def test_threaded_equals_single_call(oracle_mod):
    b = _batch()
    full = oracle.paged_attention(b.pool, b.n_pages, b.page_elems, b.bs, b.Hkv, b.d, b.q, b.table, b.ctx_lens,
                                  b.scale)
    for T in (1, 2, 3, 16):
        got = par_oracle.paged_attention(b.pool, b.n_pages, b.page_elems, b.bs, b.Hkv, b.d, b.q, b.table,
                                         b.ctx_lens, b.scale, threads=T)
        assert np.array_equal(got, full), T


def test_subset_rows_are_the_full_rows_and_the_rest_nan(oracle_mod):
    b = _batch()
    full = oracle.paged_attention(b.pool, b.n_pages, b.page_elems, b.bs, b.Hkv, b.d, b.q, b.table, b.ctx_lens,
                                  b.scale)
    ids = np.array([7, 0, 4], np.int32)
    for T in (1, 2):
        got = par_oracle.paged_attention(b.pool, b.n_pages, b.page_elems, b.bs, b.Hkv, b.d, b.q, b.table,
                                         b.ctx_lens, b.scale, seq_ids=ids, threads=T)
        assert np.array_equal(got[ids], full[ids])
        rest = np.setdiff1d(np.arange(b.S), ids)
        assert np.isnan(got[rest]).all()
    # an empty sequence (n = 0) gives zeros, in a subset too
    lens = b.ctx_lens.copy()
    lens[3] = 0
    z = oracle.paged_attention(b.pool, b.n_pages, b.page_elems, b.bs, b.Hkv, b.d, b.q, b.table, lens,
                               b.scale, seq_ids=np.array([3], np.int32))
    assert (z[3] == 0).all()
