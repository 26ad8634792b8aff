"""GPU parity: the CUDA path (through the C ABI) against the fp64 oracle on
the same seeded inputs.

Bars: the pool after append and everything indexed through the block table
bit-exact; attention max |err| <= 1.5e-2 and mean |err| <= 2e-3 against the
oracle's fp64 result (bf16 out, fp32 accumulate).
"""
import numpy as np
import pytest

import oracle
from paper_2606_12950_gb300 import workloads as W

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

MAX_ABS = 1.5e-2
MEAN_ABS = 2e-3
VARIANTS = [1, 2]  # CUDA-core FMA, tensor-core MMA


@pytest.fixture(scope="module", autouse=True)
def _cuda():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2606_12950_gb300 import runner  # noqa: F401  (builds/loads libkvpool)


def run(b, variant, num_splits=0, pool_u16=None, fused=False):
    from paper_2606_12950_gb300.runner import DeviceBatch, DevicePool

    pool = DevicePool(b.n_pages, b.page_elems * 2, b.bs, [(b.Hkv, b.d)])
    pool.upload(b.pool if pool_u16 is None else pool_u16)
    pool.set_variant(variant)
    db = DeviceBatch(pool, 0, b, num_splits)
    if fused:
        db.append_attend()
    else:
        db.append()
        db.attend()
    torch.cuda.synchronize()
    return pool, db


def check_attention(got, ref, what=""):
    err = np.abs(got - ref)
    assert np.isfinite(got).all(), f"{what}: non-finite output"
    assert err.max() <= MAX_ABS, f"{what}: max abs err {err.max():.3e}"
    assert err.mean() <= MEAN_ABS, f"{what}: mean abs err {err.mean():.3e}"
    return err


@pytest.mark.parametrize("fused", [False, True], ids=["separate", "fused"])
@pytest.mark.parametrize("variant", VARIANTS)
@pytest.mark.parametrize("num_splits", [0, 1, 3, 64])
def test_config1_append_and_attention(variant, num_splits, fused):
    b = W.config1_tiny()
    pool, db = run(b, variant, num_splits, fused=fused)
    ref_pool = oracle.batch_append(b)
    assert np.array_equal(pool.download(), ref_pool), "pool after append differs"
    ref = oracle.batch_attention(b, pool=ref_pool)
    check_attention(db.out_f64(), ref, f"config1 v{variant} splits{num_splits}")
    assert pool.error() == 0


SHAPES = [
    # (G, Hkv, d, bs, pre-append lengths)
    (1, 4, 128, 16, [0, 14, 15, 16, 30, 31, 47, 200]),
    (2, 2, 64, 16, [1, 16, 33, 700]),
    (4, 2, 128, 32, [31, 32, 63, 64, 95, 1000, 3]),
    (5, 2, 128, 16, [5, 17, 250, 1500]),
    (8, 1, 128, 16, [9, 77, 400]),
    (4, 8, 64, 32, [100, 2, 33]),
]


@pytest.mark.parametrize("fused", [False, True], ids=["separate", "fused"])
@pytest.mark.parametrize("variant", VARIANTS)
@pytest.mark.parametrize("shape", SHAPES, ids=lambda s: f"G{s[0]}_Hkv{s[1]}_d{s[2]}_bs{s[3]}")
def test_shapes_against_oracle(variant, shape, fused):
    G, Hkv, d, bs, lens = shape
    if variant == 1 and G == 8:
        pytest.skip("the CUDA-core variant is built for G <= 5")
    b = W.make_batch(500 + G * 7 + d + bs, lens, Hq=G * Hkv, Hkv=Hkv, d=d, bs=bs, extra_blocks=9)
    pool, db = run(b, variant, fused=fused)
    ref_pool = oracle.batch_append(b)
    assert np.array_equal(pool.download(), ref_pool)
    ref = oracle.batch_attention(b, pool=ref_pool)
    check_attention(db.out_f64(), ref, f"{shape} v{variant}")
    assert pool.error() == 0


@pytest.mark.parametrize("variant", VARIANTS)
def test_garbage_past_the_context_does_not_leak(variant):
    """Rows after the last token of a block hold NaN bit patterns: the
    output must not see them (P is zero there, and the MMA path clears them)."""
    b = W.make_batch(77, [3, 20, 45], Hq=8, Hkv=2, d=128, bs=32, extra_blocks=4)
    pool_u16 = b.pool.copy()
    view = pool_u16.reshape(b.n_pages, 2, b.Hkv, b.bs, b.d)
    for s in range(b.S):
        n = int(b.ctx_lens[s])
        last = b.table[s, (n - 1) // b.bs]
        view[last, :, :, n % b.bs if n % b.bs else b.bs:, :] = 0xFFFF  # NaN
    b.pool = pool_u16
    pool, db = run(b, variant, pool_u16=pool_u16)
    ref_pool = oracle.batch_append(b)
    assert np.array_equal(pool.download(), ref_pool)
    check_attention(db.out_f64(), oracle.batch_attention(b, pool=ref_pool), "NaN tail")


@pytest.mark.parametrize("variant", VARIANTS)
def test_block_placement_does_not_change_bits(variant):
    b = W.make_batch(91, [40, 300, 1200, 17], Hq=16, Hkv=4, d=128, bs=16, extra_blocks=50)
    _, db1 = run(b, variant)
    out1 = db1.out_bits()
    rng = np.random.default_rng(3)
    perm = rng.permutation(b.n_pages)
    blocks = b.pool.reshape(b.n_pages, b.page_elems)
    pool2 = np.empty_like(blocks)
    pool2[perm] = blocks
    b2 = W.make_batch(91, [40, 300, 1200, 17], Hq=16, Hkv=4, d=128, bs=16, extra_blocks=50, fill_pool=False)
    b2.pool = pool2.reshape(-1)
    b2.table = np.where(b.table >= 0, perm[np.maximum(b.table, 0)], -1).astype(np.int32)
    _, db2 = run(b2, variant)
    assert np.array_equal(out1, db2.out_bits())


@pytest.mark.parametrize("variant", VARIANTS)
def test_split_counts_agree(variant):
    b = W.make_batch(92, [5000, 33, 2047, 900, 1], Hq=32, Hkv=8, d=128, bs=16, extra_blocks=3)
    ref_pool = oracle.batch_append(b)
    ref = oracle.batch_attention(b, pool=ref_pool)
    outs = []
    for ns in [1, 2, 5, 16, 100, 0]:
        _, db = run(b, variant, ns)
        outs.append(db.out_f64())
        check_attention(outs[-1], ref, f"splits={ns}")
    base = outs[0]
    for o in outs[1:]:
        # same math in another order: within a couple of bf16 ulps of the unsplit result
        assert np.all(np.abs(o - base) <= 2.0 ** -6 * np.abs(base) + 2e-3)


def test_empty_batch_and_empty_sequences():
    b = W.make_batch(93, [10, 50], Hq=8, Hkv=2, d=64, bs=16, extra_blocks=2)
    pool, db = run(b, 2)
    lens = b.ctx_lens.copy()
    lens[0] = 0
    db.upload_table(b.table, lens)
    db.out.fill_(1.0)
    db.attend()
    torch.cuda.synchronize()
    out = db.out_f64()
    assert np.all(out[0] == 0.0)
    b.ctx_lens = lens
    check_attention(out[1:], oracle.batch_attention(b, pool=pool.download())[1:], "with empty seq")


@pytest.mark.parametrize("variant", VARIANTS)
def test_device_bounds_check_sets_error_word(variant):
    """A table entry outside the pool, planted directly in device memory
    (bypassing the host check), is skipped by both kernels and reported."""
    b = W.make_batch(94, [20, 40], Hq=8, Hkv=2, d=128, bs=16, extra_blocks=2)
    pool, db = run(b, variant)
    assert pool.error() == 0
    before = pool.download()
    bad = db.table.clone()
    bad[1, 0] = b.n_pages + 5
    db.table.copy_(bad)
    db.append()
    db.attend()
    torch.cuda.synchronize()
    assert pool.error() == -4
    assert np.array_equal(pool.download(), before)  # sequence 0 rewrote the same bytes
    assert pool.error() == 0  # read-and-clear


@pytest.mark.parametrize("fused", [False, True], ids=["separate", "fused"])
@pytest.mark.parametrize("variant", VARIANTS)
def test_decode_steps_track_the_oracle(variant, fused):
    """Several append+attend steps with growing lengths (including block
    boundaries), fresh q/k/v each step."""
    b = W.make_batch(95, [14, 15, 31, 47], Hq=8, Hkv=2, d=128, bs=16, table_tokens=np.array([64] * 4))
    from paper_2606_12950_gb300.runner import DeviceBatch, DevicePool

    pool = DevicePool(b.n_pages, b.page_elems * 2, b.bs, [(b.Hkv, b.d)])
    pool.upload(b.pool)
    pool.set_variant(variant)
    db = DeviceBatch(pool, 0, b)
    host_pool = b.pool.copy()
    lens = b.ctx_lens.copy()
    for step in range(5):
        q, kn, vn = W.step_rows(95, step, b.S, b.Hq, b.Hkv, b.d)
        db.set_rows(q, kn, vn)
        db.upload_table(b.table, lens)
        if fused:
            db.append_attend()
        else:
            db.append()
            db.attend()
        torch.cuda.synchronize()
        host_pool = oracle.append(host_pool, b.n_pages, b.page_elems, b.bs, b.Hkv, b.d, kn, vn, b.table, lens)
        ref = oracle.paged_attention(host_pool, b.n_pages, b.page_elems, b.bs, b.Hkv, b.d, q, b.table, lens,
                                     b.scale)
        check_attention(db.out_f64(), ref, f"step {step}")
        lens = lens + 1
    assert np.array_equal(pool.download(), host_pool)


@pytest.mark.parametrize("fused", [False, True], ids=["separate", "fused"])
@pytest.mark.parametrize("variant", VARIANTS)
def test_llama8b_layer_full_size(variant, fused):
    """The Llama-3-8B-shaped layer (64 sequences, 32 q / 8 KV heads, d=128,
    bs=16, lognormal lengths) at full size in the benchmark's launch
    configuration, every sequence against the oracle."""
    b = W.config2_llama8b()
    pool, db = run(b, variant, fused=fused)
    ref_pool = oracle.batch_append(b)
    got_pool = pool.download()
    assert np.array_equal(got_pool, ref_pool)
    ref = oracle.batch_attention(b, pool=ref_pool)
    check_attention(db.out_f64(), ref, f"llama8b v{variant}")
    assert pool.error() == 0
