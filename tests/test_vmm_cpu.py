"""Host bookkeeping of the VMM-backed elastic pool (kv_pool_create_vmm,
kv_pool_trim, kv_budget_*) with a caller-supplied fake backing, so no GPU is
needed: chunks are mapped on demand by kv_alloc_blocks (all-or-nothing),
limits and a shared budget reject requests with KV_ERR_OUT_OF_BLOCKS, and
trim returns whole free superpages and unmaps whole free chunks (§III-C)."""
import numpy as np
import pytest

from paper_2606_12950_gb300 import kvpool as K

FAKE_BASE = 1 << 40
FAKE_ERR = (1 << 40) - 4096
BLOCK = 2 * 8 * 16 * 128 * 2  # 8 KV heads, bs 16, d 128: 64 KiB


class FakeBacking:
    def __init__(self, fail_after=None):
        self.mapped = {}
        self.calls = 0
        self.fail_after = fail_after

    def map(self, off, n):
        self.calls += 1
        if self.fail_after is not None and len(self.mapped) >= self.fail_after:
            return 1
        assert off not in self.mapped
        self.mapped[off] = n
        return 0

    def unmap(self, off, n):
        assert self.mapped.pop(off) == n
        return 0


def make(virtual_chunks=16, chunk=4 * BLOCK, layouts=((8, 128),), limit=0, budget=None, backing=None, seed=0):
    backing = backing or FakeBacking()
    p = K.kv_pool_create_vmm(virtual_chunks * chunk, 16, list(layouts), FAKE_ERR, chunk_bytes=chunk,
                             physical_limit=limit, budget=budget, backend=backing, device_base=FAKE_BASE,
                             shuffle_seed=seed)
    return p, backing


def chunk_of(ids, chunk=4 * BLOCK):
    return set(int(i) * BLOCK // chunk for i in np.atleast_1d(ids))


def test_nothing_is_mapped_until_blocks_are_allocated():
    p, fb = make()
    st = K.kv_pool_stats(p)
    assert st["bytes_mapped"] == 0 and fb.mapped == {}
    assert st["blocks_capacity"][0] == 16 * 4  # the virtual capacity
    ids = K.kv_alloc_blocks(p, 0, 5)  # two chunks of four blocks
    assert len(fb.mapped) == 2 and K.kv_pool_stats(p)["bytes_mapped"] == 2 * 4 * BLOCK
    assert {o // (4 * BLOCK) for o in fb.mapped} == chunk_of(ids)
    ids2 = K.kv_alloc_blocks(p, 0, 3)  # fits the mapped chunks
    assert len(fb.mapped) == 2 and not (set(ids) & set(ids2))
    K.kv_pool_destroy(p)
    assert fb.mapped == {}  # destroy unmaps everything


def test_physical_limit_rejects_whole_request():
    p, fb = make(limit=3 * 4 * BLOCK)
    K.kv_alloc_blocks(p, 0, 10)  # 3 chunks
    before = K.kv_pool_stats(p)
    with pytest.raises(K.KVError) as e:
        K.kv_alloc_blocks(p, 0, 3)  # needs a 4th chunk
    assert e.value.code == K.KV_ERR_OUT_OF_BLOCKS
    after = K.kv_pool_stats(p)
    assert after["blocks_used"] == before["blocks_used"] and after["bytes_mapped"] == before["bytes_mapped"]
    K.kv_alloc_blocks(p, 0, 2)  # the mapped chunks still have room for 2
    K.kv_pool_destroy(p)


def test_backing_failure_is_out_of_blocks_and_allocates_nothing():
    fb = FakeBacking(fail_after=2)
    p, _ = make(backing=fb)
    with pytest.raises(K.KVError) as e:
        K.kv_alloc_blocks(p, 0, 9)  # needs 3 chunks, the third fails
    assert e.value.code == K.KV_ERR_OUT_OF_BLOCKS
    st = K.kv_pool_stats(p)
    assert st["blocks_used"][0] == 0 and st["bytes_mapped"] == 2 * 4 * BLOCK  # mapped chunks stay as capacity
    assert len(K.kv_alloc_blocks(p, 0, 8)) == 8
    K.kv_pool_destroy(p)


def test_trim_unmaps_whole_free_chunks_only():
    p, fb = make()
    a = K.kv_alloc_blocks(p, 0, 8)   # chunks 0, 1 (ascending order)
    b = K.kv_alloc_blocks(p, 0, 4)   # chunk 2
    assert K.kv_pool_trim(p) == 0    # nothing free
    K.kv_free_blocks(p, 0, a[:6])    # chunk 0 fully free, chunk 1 half
    released = K.kv_pool_trim(p)
    assert released == 4 * BLOCK and len(fb.mapped) == 2
    assert chunk_of(a[6:]) | chunk_of(b) == {o // (4 * BLOCK) for o in fb.mapped}
    st = K.kv_pool_stats(p)
    assert st["blocks_used"][0] == 6 and st["bytes_mapped"] == 2 * 4 * BLOCK
    K.kv_free_blocks(p, 0, a[6:])
    K.kv_free_blocks(p, 0, b)
    assert K.kv_pool_trim(p) == 2 * 4 * BLOCK and fb.mapped == {}
    # everything can be mapped again
    assert len(K.kv_alloc_blocks(p, 0, 64)) == 64 and len(fb.mapped) == 16
    K.kv_pool_destroy(p)


def test_shared_budget_across_pools():
    """Two pools each reserve 16 chunks (8x the budget together); the budget
    of 4 chunks bounds what both map; trimming one lets the other grow."""
    bud = K.kv_budget_create(4 * 4 * BLOCK)
    p1, f1 = make(budget=bud)
    p2, f2 = make(budget=bud)
    x = K.kv_alloc_blocks(p1, 0, 12)
    K.kv_alloc_blocks(p2, 0, 4)
    assert K.kv_budget_used(bud) == 4 * 4 * BLOCK
    with pytest.raises(K.KVError):
        K.kv_alloc_blocks(p2, 0, 5)  # a fifth chunk would exceed the budget
    K.kv_free_blocks(p1, 0, x)
    assert K.kv_budget_used(bud) == 4 * 4 * BLOCK  # freed blocks stay mapped until trim
    assert K.kv_pool_trim(p1) == 3 * 4 * BLOCK
    assert K.kv_budget_used(bud) == 4 * BLOCK
    K.kv_alloc_blocks(p2, 0, 12)
    assert K.kv_budget_used(bud) == 4 * 4 * BLOCK
    with pytest.raises(K.KVError):
        K.kv_budget_destroy(bud)  # still in use
    K.kv_pool_destroy(p1)
    K.kv_pool_destroy(p2)
    assert K.kv_budget_used(bud) == 0
    K.kv_budget_destroy(bud)


def test_trim_moves_free_superpages_between_layouts():
    """MHA blocks are 4 pages of the GQA block size: after the MHA layout
    frees everything, trim hands its superpages back and the GQA layout can
    carve them (a fixed pool behaves the same)."""
    layouts = ((8, 128), (32, 128))
    p, fb = make(virtual_chunks=2, chunk=8 * BLOCK, layouts=layouts)
    big = K.kv_alloc_blocks(p, 1, 4)  # 4 superpages = both chunks
    with pytest.raises(K.KVError):
        K.kv_alloc_blocks(p, 0, 1)
    K.kv_free_blocks(p, 1, big)
    with pytest.raises(K.KVError):
        K.kv_alloc_blocks(p, 0, 1)  # still carved for the MHA layout
    released = K.kv_pool_trim(p)
    assert released == 2 * 8 * BLOCK and fb.mapped == {}
    assert len(K.kv_alloc_blocks(p, 0, 16)) == 16
    K.kv_pool_destroy(p)


def test_random_ops_keep_mapping_invariants():
    """Random alloc / free / trim: every live block lies in a mapped chunk;
    bytes_mapped = mapped chunks x chunk; after a trim no mapped chunk is
    wholly free; the fake backing agrees with the library's accounting."""
    rng = np.random.default_rng(5)
    chunk = 4 * BLOCK
    p, fb = make(virtual_chunks=24, chunk=chunk, limit=20 * chunk, seed=9)
    live = []
    for it in range(800):
        op = rng.integers(0, 10)
        if op < 5:
            n = int(rng.integers(1, 12))
            try:
                live += list(K.kv_alloc_blocks(p, 0, n))
            except K.KVError as e:
                assert e.code == K.KV_ERR_OUT_OF_BLOCKS
        elif op < 9 and live:
            k = int(rng.integers(1, len(live) + 1))
            idx = rng.choice(len(live), size=k, replace=False)
            K.kv_free_blocks(p, 0, [live[i] for i in idx])
            live = [b for j, b in enumerate(live) if j not in set(idx.tolist())]
        else:
            K.kv_pool_trim(p)
            used_chunks = chunk_of(live, chunk) if live else set()
            assert {o // chunk for o in fb.mapped} == used_chunks
        st = K.kv_pool_stats(p)
        assert st["blocks_used"][0] == len(live)
        assert st["bytes_mapped"] == len(fb.mapped) * chunk <= 20 * chunk
        if live:
            assert chunk_of(live, chunk) <= {o // chunk for o in fb.mapped}
    K.kv_pool_destroy(p)


def test_argument_checks():
    with pytest.raises(K.KVError):  # a caller backing needs a chunk size
        K.kv_pool_create_vmm(1 << 24, 16, [(8, 128)], FAKE_ERR, chunk_bytes=0, backend=FakeBacking(),
                             device_base=FAKE_BASE)
    with pytest.raises(K.KVError):  # limit below one chunk
        make(limit=BLOCK)
    p, _ = make(virtual_chunks=3)
    assert K.kv_pool_get_base(p) == FAKE_BASE
    assert K.kv_pool_stats(p)["pages_total"] == 3 * 4
    K.kv_pool_destroy(p)
