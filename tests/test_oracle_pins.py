"""Pins for the fp64 oracle, independent of the oracle itself.

Each check ties the oracle to something it does not compute on its own:
a dense brute force written against a separate numpy gather, PyTorch's CPU
fp64 scaled-dot-product attention (a library special case), closed forms of
softmax attention, exact invariances of the definition, and a hand-derived
two-token example (tests/golden/).  Together they fail on a dropped scale, a
wrong sign, a wrong head group, a wrong slot/offset index, a transposed K/V,
or an off-by-one context length.
"""
import json
import math
import os

import numpy as np
import pytest

from paper_2606_12950_gb300 import workloads as W

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def gather_dense(b, pool):
    """Numpy gather of each sequence's K/V in logical order: list of
    (K [Hkv, n, d], V [Hkv, n, d]) as fp64.  Uses array reshapes, not the
    oracle's accessor."""
    blocks = pool[: (pool.size // b.page_elems) * b.page_elems].reshape(-1, b.page_elems)
    out = []
    for s in range(b.S):
        n = int(b.ctx_lens[s])
        nb = (n + b.bs - 1) // b.bs
        ids = b.table[s, :nb]
        blk = blocks[ids, : b.block_elems].reshape(nb, 2, b.Hkv, b.bs, b.d)
        # [nb, Hkv, bs, d] -> [Hkv, nb*bs, d] -> first n positions
        K = blk[:, 0].transpose(1, 0, 2, 3).reshape(b.Hkv, nb * b.bs, b.d)[:, :n]
        V = blk[:, 1].transpose(1, 0, 2, 3).reshape(b.Hkv, nb * b.bs, b.d)[:, :n]
        out.append((W.bf16_bits_to_f64(K), W.bf16_bits_to_f64(V)))
    return out


def numpy_attention(q, K, V, scale):
    """Plain numpy softmax attention, heads grouped contiguously."""
    Hq = q.shape[0]
    Hkv = K.shape[0]
    G = Hq // Hkv
    o = np.zeros_like(q)
    for h in range(Hq):
        g = h // G
        x = scale * (K[g] @ q[h])
        p = np.exp(x - x.max())
        p /= p.sum()
        o[h] = p @ V[g]
    return o


def tiny_random(seed, lens, Hq=4, Hkv=2, d=16, bs=4, extra=5):
    b = W.make_batch(seed, np.asarray(lens) - 1, Hq=Hq, Hkv=Hkv, d=d, bs=bs, extra_blocks=extra)
    return b


CASES = [
    (11, [1, 3, 4, 5, 8, 9], 4, 2, 16, 4),
    (12, [2, 7, 33], 8, 2, 32, 8),
    (13, [5, 16, 17], 3, 3, 8, 16),  # MHA
    (14, [40, 1], 5, 1, 8, 4),  # MQA, G=5
]


@pytest.mark.parametrize("seed,lens,Hq,Hkv,d,bs", CASES)
def test_paged_equals_dense_brute_force(oracle_mod, seed, lens, Hq, Hkv, d, bs):
    b = tiny_random(seed, lens, Hq, Hkv, d, bs)
    got = oracle_mod.batch_attention(b)
    dense = gather_dense(b, b.pool)
    for s, (K, V) in enumerate(dense):
        q = W.bf16_bits_to_f64(b.q[s])
        ref_c = oracle_mod.dense_attention(q, K, V, b.scale)
        ref_np = numpy_attention(q, K, V, b.scale)
        np.testing.assert_allclose(got[s], ref_c, rtol=0, atol=1e-12)
        np.testing.assert_allclose(got[s], ref_np, rtol=0, atol=1e-12)


def test_config1_matches_torch_sdpa(oracle_mod):
    torch = pytest.importorskip("torch")
    import torch.nn.functional as F

    b = W.config1_tiny()
    pool = oracle_mod.batch_append(b)
    got = oracle_mod.batch_attention(b, pool=pool)
    for s, (K, V) in enumerate(gather_dense(b, pool)):
        q = torch.from_numpy(W.bf16_bits_to_f64(b.q[s]))[None, :, None, :]  # [1, Hq, 1, d]
        k = torch.from_numpy(K)[None]
        v = torch.from_numpy(V)[None]
        ref = F.scaled_dot_product_attention(q, k, v, scale=b.scale, enable_gqa=True)[0, :, 0]
        np.testing.assert_allclose(got[s], ref.numpy(), rtol=0, atol=1e-12)


def test_one_token_returns_v0_exactly(oracle_mod):
    b = tiny_random(21, [1, 1, 1], Hq=4, Hkv=2, d=8, bs=4)
    got = oracle_mod.batch_attention(b)
    for s, (K, V) in enumerate(gather_dense(b, b.pool)):
        for h in range(b.Hq):
            assert np.array_equal(got[s, h], V[h // b.G, 0])


def _set_rows(b, pool, s, g, which, rows):
    """Write rows [n, d] (bf16 bits) into K (which=0) or V (which=1) of (s, g)
    through a numpy view of the layout."""
    blocks = pool.reshape(-1, b.page_elems)
    for j, row in enumerate(rows):
        blk = b.table[s, j // b.bs]
        view = blocks[blk, : b.block_elems].reshape(2, b.Hkv, b.bs, b.d)
        view[which, g, j % b.bs] = row


def test_identical_keys_give_mean_of_v(oracle_mod):
    b = tiny_random(22, [9, 13], Hq=4, Hkv=2, d=8, bs=4)
    pool = b.pool.copy()
    rng = np.random.default_rng(5)
    for s in range(b.S):
        n = int(b.ctx_lens[s])
        for g in range(b.Hkv):
            key = W.bf16_normal(rng, (b.d,))
            _set_rows(b, pool, s, g, 0, [key] * n)
    got = oracle_mod.batch_attention(b, pool=pool)
    for s, (K, V) in enumerate(gather_dense(b, pool)):
        for h in range(b.Hq):
            np.testing.assert_allclose(got[s, h], V[h // b.G].mean(axis=0), rtol=0, atol=1e-13)


def test_zero_query_gives_mean_of_v(oracle_mod):
    b = tiny_random(23, [7, 20], Hq=2, Hkv=1, d=8, bs=4)
    b.q[:] = 0
    got = oracle_mod.batch_attention(b)
    for s, (K, V) in enumerate(gather_dense(b, b.pool)):
        for h in range(b.Hq):
            np.testing.assert_allclose(got[s, h], V[0].mean(axis=0), rtol=0, atol=1e-13)


def test_dominant_key_selects_its_value(oracle_mod):
    b = tiny_random(24, [12], Hq=2, Hkv=1, d=8, bs=4)
    pool = b.pool.copy()
    n = int(b.ctx_lens[0])
    # q = e_0 (bf16 1.0 = 0x3F80); keys zero except key 5 has component 0 = 64
    b.q[:] = 0
    b.q[0, :, 0] = 0x3F80
    keys = np.zeros((n, b.d), np.uint16)
    keys[5, 0] = W.bf16_bits_from_f32(np.array([64.0], np.float32))[0]
    _set_rows(b, pool, 0, 0, 0, keys)
    got = oracle_mod.batch_attention(b, pool=pool)
    V = gather_dense(b, pool)[0][1][0]
    # weight of key 5: e^(64*s) / (e^(64*s) + n-1) with s = 1/sqrt(8)
    x = 64.0 * b.scale
    p5 = math.exp(x) / (math.exp(x) + (n - 1))
    expect = p5 * V[5] + (1 - p5) / (n - 1) * (V.sum(axis=0) - V[5])
    np.testing.assert_allclose(got[0, 0], expect, rtol=0, atol=1e-12)
    np.testing.assert_allclose(got[0, 0], V[5], rtol=0, atol=1e-6)


def test_golden_two_token_example(oracle_mod):
    """Hand-derived example (tests/golden/two_token.json)."""
    with open(os.path.join(GOLDEN, "two_token.json")) as f:
        g = json.load(f)
    q = np.array(g["q"], np.float64)
    k = np.array(g["k"], np.float64)
    v = np.array(g["v"], np.float64)
    out = oracle_mod.dense_attention(q, k, v, g["scale"])
    np.testing.assert_allclose(out, np.array(g["expected"]), rtol=0, atol=1e-15)
    # the same numbers through the paged path: put the two tokens in two
    # one-token blocks, stored in reverse physical order
    d = q.shape[1]
    bits = lambda a: W.bf16_bits_from_f32(np.asarray(a, np.float32))
    page = 2 * 1 * 1 * d
    pool = np.zeros(2 * page, np.uint16)
    pool[page * 1 : page * 1 + d] = bits(k[0, 0])
    pool[page * 1 + d : page * 2] = bits(v[0, 0])
    pool[0:d] = bits(k[0, 1])
    pool[d : 2 * d] = bits(v[0, 1])
    table = np.array([[1, 0]], np.int32)
    qb = bits(q)[None]
    got = oracle_mod.paged_attention(pool, 2, page, 1, 1, d, qb, table, np.array([2], np.int32), g["scale"])
    np.testing.assert_allclose(got[0], np.array(g["expected"]), rtol=0, atol=1e-15)


def test_block_permutation_invariance_is_exact(oracle_mod):
    b = W.config1_tiny()
    base = oracle_mod.batch_attention(b)
    rng = np.random.default_rng(99)
    perm = rng.permutation(b.n_pages)  # new id of old block i
    blocks = b.pool.reshape(b.n_pages, b.page_elems)
    pool2 = np.empty_like(blocks)
    pool2[perm] = blocks
    table2 = np.where(b.table >= 0, perm[np.maximum(b.table, 0)], -1).astype(np.int32)
    got = oracle_mod.paged_attention(pool2.reshape(-1), b.n_pages, b.page_elems, b.bs, b.Hkv, b.d,
                                     b.q, table2, b.ctx_lens, b.scale)
    assert np.array_equal(base, got)


@pytest.mark.parametrize("split_len", [1, 3, 16, 17, 64, 1000])
def test_split_combine_equals_unsplit(oracle_mod, split_len):
    b = W.config1_tiny()
    full = oracle_mod.batch_attention(b)
    split = oracle_mod.split_attention(b.pool, b.n_pages, b.page_elems, b.bs, b.Hkv, b.d, b.q,
                                       b.table, b.ctx_lens, b.scale, split_len)
    np.testing.assert_allclose(split, full, rtol=0, atol=1e-13)


@pytest.mark.parametrize("seed,lens,Hq,Hkv,d,bs", CASES)
@pytest.mark.parametrize("split_len", [1, 2, 5, 16])
def test_split_attention_equals_dense_brute_force(oracle_mod, seed, lens, Hq, Hkv, d, bs, split_len):
    """The split-K form (per-split partials, then the combine step) pinned
    directly to the numpy gather and softmax, not only to the unsplit
    oracle: a wrong rescale between splits, a dropped split or a merge in
    the wrong order fails here."""
    b = tiny_random(seed, lens, Hq, Hkv, d, bs)
    got = oracle_mod.split_attention(b.pool, b.n_pages, b.page_elems, b.bs, b.Hkv, b.d, b.q,
                                     b.table, b.ctx_lens, b.scale, split_len)
    for s, (K, V) in enumerate(gather_dense(b, b.pool)):
        q = W.bf16_bits_to_f64(b.q[s])
        np.testing.assert_allclose(got[s], numpy_attention(q, K, V, b.scale), rtol=0, atol=1e-12)


@pytest.mark.parametrize("split_len", [1, 3, 4])
def test_split_attention_with_identical_keys_gives_mean_of_v(oracle_mod, split_len):
    """Closed form through the split path: equal keys make every score equal,
    so each split's partial and their merge must give the plain mean of V."""
    b = tiny_random(25, [9, 13], Hq=4, Hkv=2, d=8, bs=4)
    pool = b.pool.copy()
    rng = np.random.default_rng(6)
    for s in range(b.S):
        n = int(b.ctx_lens[s])
        for g in range(b.Hkv):
            _set_rows(b, pool, s, g, 0, [W.bf16_normal(rng, (b.d,))] * n)
    got = oracle_mod.split_attention(pool, b.n_pages, b.page_elems, b.bs, b.Hkv, b.d, b.q, b.table,
                                     b.ctx_lens, b.scale, split_len)
    for s, (K, V) in enumerate(gather_dense(b, pool)):
        for h in range(b.Hq):
            np.testing.assert_allclose(got[s, h], V[h // b.G].mean(axis=0), rtol=0, atol=1e-13)


@pytest.mark.parametrize("seed,lens,Hq,Hkv,d,bs", CASES)
def test_sequence_subset_equals_dense_brute_force(oracle_mod, seed, lens, Hq, Hkv, d, bs):
    """The seq_ids subset path pinned directly: the requested sequences'
    rows equal the numpy gather and softmax, every other row stays NaN, and
    the order of the ids does not matter."""
    b = tiny_random(seed, lens, Hq, Hkv, d, bs)
    ids = np.array([s for s in range(b.S) if s % 2 == 1][::-1] + [0], dtype=np.int32)
    got = oracle_mod.paged_attention(b.pool, b.n_pages, b.page_elems, b.bs, b.Hkv, b.d, b.q, b.table,
                                     b.ctx_lens, b.scale, seq_ids=ids)
    dense = gather_dense(b, b.pool)
    for s in range(b.S):
        if s in set(ids.tolist()):
            K, V = dense[s]
            q = W.bf16_bits_to_f64(b.q[s])
            np.testing.assert_allclose(got[s], numpy_attention(q, K, V, b.scale), rtol=0, atol=1e-12)
        else:
            assert np.isnan(got[s]).all()


def test_append_writes_exactly_the_new_slot(oracle_mod):
    b = W.make_batch(31, [17, 64, 100, 255, 0], Hq=4, Hkv=2, d=64, bs=16, n_pages=128,
                     pool_fill="sentinel")
    after = oracle_mod.batch_append(b)
    # replay the slot formula by brute force over every pool element
    expect = np.full_like(b.pool, 0xFFFF)
    for s in range(b.S):
        pos = int(b.ctx_lens[s]) - 1
        blk = int(b.table[s, pos // b.bs])
        off = pos % b.bs
        for g in range(b.Hkv):
            for c in range(b.d):
                base = blk * b.page_elems
                expect[base + ((0 * b.Hkv + g) * b.bs + off) * b.d + c] = b.k_new[s, g, c]
                expect[base + ((1 * b.Hkv + g) * b.bs + off) * b.d + c] = b.v_new[s, g, c]
    assert np.array_equal(after, expect)
    assert int((after != 0xFFFF).sum()) <= 2 * b.S * b.Hkv * b.d


def test_empty_sequence_gives_zero(oracle_mod):
    b = tiny_random(41, [3, 5], Hq=2, Hkv=1, d=8, bs=4)
    b.ctx_lens = np.array([0, 5], np.int32)
    got = oracle_mod.batch_attention(b)
    assert np.all(got[0] == 0.0)


def test_out_of_pool_index_is_rejected(oracle_mod):
    b = tiny_random(42, [3, 5], Hq=2, Hkv=1, d=8, bs=4)
    b.table[1, 0] = b.n_pages  # one past the end
    with pytest.raises(ValueError):
        oracle_mod.batch_attention(b)
    with pytest.raises(ValueError):
        oracle_mod.batch_append(b.__class__(**{**b.__dict__, "ctx_lens": np.array([3, 1], np.int32)}))


def test_generator_bf16_rounding_is_rne():
    x = np.array([1.0, 1.00390625, 1.01171875, -2.0, 3.0e-3, 1.0 + 2 ** -8 + 2 ** -20], np.float32)
    # 1+2^-8 is a tie between 1.0 and 1+2^-7 -> even (1.0); 1+3*2^-8 ties -> 1+2^-6 (even)
    bits = W.bf16_bits_from_f32(x)
    assert bits[0] == 0x3F80
    assert bits[1] == 0x3F80
    assert bits[2] == 0x3F82
    assert bits[3] == 0xC000
    assert bits[5] == 0x3F81  # just above the tie rounds up
    back = W.bf16_bits_to_f64(bits)
    assert abs(back[4] - 3.0e-3) <= 2 ** -8 * 3.0e-3  # half an ulp of an 8-bit significand


def test_generator_is_seeded_and_shaped():
    a = W.config1_tiny()
    b = W.config1_tiny()
    assert np.array_equal(a.pool, b.pool) and np.array_equal(a.table, b.table)
    assert list(a.ctx_lens) == [18, 65, 101, 256]
    used = a.table[a.table >= 0]
    assert len(set(used.tolist())) == used.size  # no block used twice
    assert used.max() < 128
