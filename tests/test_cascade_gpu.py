"""GPU parity of shared-prefix (cascade) decode attention through the C ABI
(paged_decode_attn_cascade) against the fp64 oracle.

The oracle knows nothing of the cascade: it evaluates the plain definition
over each sequence's block table, in which the members of a group hold the
same physical blocks for the shared prefix.  Bars as for paged attention:
max |err| <= 1.5e-2, mean |err| <= 2e-3; the pool after the fused append
bit-exact.
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


def check(got, ref, what):
    err = np.abs(got - ref)
    assert np.isfinite(got).all(), what
    assert err.max() <= MAX_ABS, f"{what}: max abs err {err.max():.3e}"
    assert err.mean() <= MEAN_ABS, f"{what}: mean abs err {err.mean():.3e}"


def build(seed, pre_lens, groups, G, Hkv, d, bs, extra_blocks=4):
    b = W.make_batch(seed, pre_lens, Hq=G * Hkv, Hkv=Hkv, d=d, bs=bs, extra_blocks=extra_blocks)
    W.share_prefix(b, groups)
    return b


def run(b, groups, fused=True, lens=None):
    from paper_2606_12950_gb300.runner import DeviceBatch, DevicePool

    pool = DevicePool(b.n_pages, b.page_elems * 2, b.bs, [(b.Hkv, b.d)])
    pool.upload(b.pool)
    db = DeviceBatch(pool, 0, b)
    if lens is not None:
        db.upload_table(b.table, lens)
    db.cascade(K.PrefixPlan(groups), fused=fused)
    torch.cuda.synchronize()
    return pool, db


SHAPES = [
    # (G, Hkv, d, bs)
    (4, 8, 128, 16),
    (1, 4, 128, 16),
    (2, 2, 64, 32),
    (5, 2, 128, 16),
    (8, 1, 128, 16),
    (4, 2, 64, 16),
]


@pytest.mark.parametrize("fused", [True, False], ids=["fused", "separate"])
@pytest.mark.parametrize("shape", SHAPES, ids=lambda s: f"G{s[0]}_Hkv{s[1]}_d{s[2]}_bs{s[3]}")
def test_two_groups_and_outsiders(shape, fused):
    """Group A: 256-token prefix, members whose suffix is 1, 44, 63, 64,
    745 and 4745 tokens (the first has only the appended token); group B:
    128-token prefix; two sequences in no group."""
    G, Hkv, d, bs = shape
    pre = [256, 300, 256 + 62, 256 + 63, 1000, 50, 128, 400, 5000, 700]
    groups = [([0, 1, 2, 3, 4, 8], 256), ([6, 7], 128)]
    b = build(4000 + G * 10 + d + bs, pre, groups, G, Hkv, d, bs)
    pool, db = run(b, groups, fused=fused)
    ref_pool = oracle.batch_append(b)
    if fused:
        assert np.array_equal(pool.download(), ref_pool), "pool after the fused append differs"
        ref = oracle.batch_attention(b, pool=ref_pool)
    else:
        ref = oracle.batch_attention(b, pool=b.pool)  # nothing appended: the pool is the input's
        assert np.array_equal(pool.download(), b.pool)
    check(db.out_f64(), ref, f"{shape} fused={fused}")
    assert pool.error() == 0


def test_member_whose_whole_context_is_the_prefix():
    """Without an append, a member of length exactly `tokens` attends over
    the prefix records alone (its suffix run is empty)."""
    pre = [191, 400, 900, 10]
    groups = [([0, 1, 2], 192)]
    b = build(4101, pre, groups, 4, 2, 128, 16)
    lens = b.ctx_lens.copy()  # post-append lengths: 192, 401, 901, 11
    pool, db = run(b, groups, fused=False, lens=lens)
    assert lens[0] == 192
    ref = oracle.batch_attention(b, pool=b.pool)
    check(db.out_f64(), ref, "prefix-only member")
    assert pool.error() == 0


@pytest.mark.parametrize("G", [1, 4, 5, 8])
def test_many_members_several_row_tiles_and_key_splits(G):
    """100 sharers of a 2048-token prefix: several 64-row tiles per KV head
    and several key splits; suffixes 1 .. 600 tokens."""
    rng = np.random.default_rng(41 + G)
    n = 100
    Hkv = 8 if G <= 4 else 2
    pre = (2048 + rng.integers(0, 600, size=n)).tolist() + [300, 2000]
    groups = [(list(range(n)), 2048)]
    b = build(4200 + G, pre, groups, G, Hkv, 128, 16)
    pool, db = run(b, groups)
    ref_pool = oracle.batch_append(b)
    assert np.array_equal(pool.download(), ref_pool)
    ids = np.array(sorted(set(rng.choice(len(pre), 24, replace=False).tolist()) | {0, n, n + 1}), np.int32)
    ref = oracle.paged_attention(ref_pool, b.n_pages, b.page_elems, b.bs, b.Hkv, b.d, b.q, b.table, b.ctx_lens,
                                 b.scale, seq_ids=ids)
    check(db.out_f64()[ids], ref[ids], f"G={G}")
    assert pool.error() == 0


def test_cascade_block_placement_does_not_change_bits():
    """Moving every physical block (prefix and suffixes) to another place in
    the pool, with the table renamed to match, gives bit-identical outputs:
    the prefix records and their merge depend only on logical positions."""
    pre = [256 + 1, 256 + 70, 256 + 700, 300, 256 + 33]
    groups = [([0, 1, 2, 4], 256)]
    b = build(4400, pre, groups, 4, 4, 128, 16, extra_blocks=40)
    _, db1 = run(b, groups)
    out1 = db1.out_bits()
    rng = np.random.default_rng(5)
    perm = rng.permutation(b.n_pages)
    blocks = b.pool.reshape(b.n_pages, b.page_elems)
    pool2 = np.empty_like(blocks)
    pool2[perm] = blocks
    b2 = build(4400, pre, groups, 4, 4, 128, 16, extra_blocks=40)
    b2.pool = pool2.reshape(-1)
    b2.table = np.where(b.table >= 0, perm[np.maximum(b.table, 0)], -1).astype(np.int32)
    _, db2 = run(b2, groups)
    assert np.array_equal(out1, db2.out_bits())


def test_prefix_grid_larger_than_half_the_gpu():
    """700 sharers at G = 4, Hkv = 8: 11 row tiles x 8 KV heads = 88 prefix
    CTAs, more than half of the SMs, so the decode grid is sized to the
    whole GPU and its CTAs start as prefix CTAs finish."""
    rng = np.random.default_rng(4300)
    n = 700
    pre = (128 + rng.integers(0, 200, size=n)).tolist() + [90, 333]
    groups = [(list(range(n)), 128)]
    b = build(4300, pre, groups, 4, 8, 128, 16)
    pool, db = run(b, groups)
    ref_pool = oracle.batch_append(b)
    assert np.array_equal(pool.download(), ref_pool)
    ids = np.array(sorted(set(rng.choice(len(pre), 24, replace=False).tolist()) | {0, n - 1, n, n + 1}), np.int32)
    ref = oracle.paged_attention(ref_pool, b.n_pages, b.page_elems, b.bs, b.Hkv, b.d, b.q, b.table, b.ctx_lens,
                                 b.scale, seq_ids=ids)
    check(db.out_f64()[ids], ref[ids], "700 sharers")
    assert pool.error() == 0


@pytest.mark.parametrize("G", [4, 5])
def test_scores_rising_inside_a_key_tile(G):
    """The prefix's keys at tokens 64..127 and 192..255 are scaled by 8, so
    the second 64-key half of each 128-key tile of the prefix kernel scores
    far above the first (by more than 2^8 in base 2): the running max rises
    inside a tile (the P already written for the tile is rescaled) and
    between tiles (O is rescaled)."""
    Hkv, d, bs = 2, 128, 16
    pre = [256 + 40, 256 + 300, 256 + 7, 900]
    groups = [([0, 1, 2], 256)]
    b = build(4500 + G, pre, groups, G, Hkv, d, bs)
    lead = groups[0][0][0]
    for j in list(range(64, 128)) + list(range(192, 256)):
        base = int(b.table[lead][j // bs]) * b.page_elems
        for g in range(Hkv):
            k0 = base + (g * bs + j % bs) * d  # K of head g at offset j % bs
            row = W.bf16_bits_to_f64(b.pool[k0:k0 + d]) * 8.0
            b.pool[k0:k0 + d] = W.bf16_bits_from_f32(row.astype(np.float32))
    pool, db = run(b, groups)
    ref_pool = oracle.batch_append(b)
    assert np.array_equal(pool.download(), ref_pool)
    ref = oracle.batch_attention(b, pool=ref_pool)
    check(db.out_f64(), ref, f"rising scores G={G}")
    assert pool.error() == 0


def test_cascade_agrees_with_plain_attention():
    """Same inputs through paged_decode_attn_append and the cascade: both
    within tolerance of the oracle and within a few bf16 ulps of each other."""
    pre = [2048 + 5, 2048 + 700, 2048 + 3000, 2048 + 16]
    groups = [([0, 1, 2, 3], 2048)]
    b = build(4300, pre, groups, 4, 8, 128, 16)
    from paper_2606_12950_gb300.runner import DeviceBatch, DevicePool

    outs = []
    for mode in ("plain", "cascade"):
        pool = DevicePool(b.n_pages, b.page_elems * 2, b.bs, [(b.Hkv, b.d)])
        pool.upload(b.pool)
        db = DeviceBatch(pool, 0, b)
        if mode == "plain":
            db.append_attend()
        else:
            db.cascade(K.PrefixPlan(groups))
        torch.cuda.synchronize()
        outs.append(db.out_f64())
    ref = oracle.batch_attention(b, pool=oracle.batch_append(b))
    for o in outs:
        check(o, ref, "plain / cascade")
    assert np.all(np.abs(outs[0] - outs[1]) <= 2.0 ** -6 * np.abs(outs[0]) + 2e-3)


def test_plan_validation():
    """Plans the library must refuse before launching anything."""
    pre = [300, 400, 500]
    b = build(4400, pre, [([0, 1, 2], 256)], 4, 2, 128, 16)
    from paper_2606_12950_gb300.runner import DeviceBatch, DevicePool

    pool = DevicePool(b.n_pages, b.page_elems * 2, b.bs, [(b.Hkv, b.d)])
    pool.upload(b.pool)
    db = DeviceBatch(pool, 0, b)
    bad = [
        [([0, 1], 100)],          # not a multiple of 64
        [([0, 1], 0)],            # empty prefix
        [([0, 1], 256), ([1, 2], 256)],  # sequence 1 in two groups
        [([0, 5], 256)],          # member out of range
        [([], 256)],              # empty group
    ]
    for groups in bad:
        with pytest.raises(K.KVError) as e:
            db.cascade(K.PrefixPlan(groups))
        assert e.value.code == K.KV_ERR_INVALID_ARG, groups
    with pytest.raises(K.KVError) as e:
        K.paged_decode_attn_cascade(pool.handle, 0, db.q, db.k_new, db.v_new, db.out, db.table, db.lens,
                                    db.max_blocks, db.S, db.Hq, b.scale, K.PrefixPlan([([0, 1], 256)]), db.ws, 256)
    assert e.value.code == K.KV_ERR_WORKSPACE
    torch.cuda.synchronize()
    assert pool.error() == 0
    assert np.array_equal(pool.download(), b.pool)  # nothing ran
