"""Host sequence tables (rows a1/a2 on the host): per-stage reservation,
one-block growth on a reservation miss, shared prefixes by reference,
release and trim, checked against the slot model in oracle/seq_model.py and
against the pool's refcounts.  No GPU: the device pointer is never touched.
"""
import numpy as np
import pytest

from oracle.seq_model import SeqModel
from paper_2606_12950_gb300 import kvpool as K

FAKE_BASE = 1 << 40
FAKE_ERR = (1 << 40) + (1 << 30)
BS = 16


def make(n_pages=400, S=12, max_blocks=40):
    pool = K.kv_pool_create(FAKE_BASE, n_pages * 65536, BS, [(8, 128)], FAKE_ERR, shuffle_seed=5)
    return pool, K.SeqTab(pool, 0, S, max_blocks)


def check_rows(t, m, pool):
    tab, lens = t.host()
    assert list(lens) == m.len
    live = {}
    for s in range(m.S):
        h = m.held[s]
        assert (tab[s, :h] >= 0).all() and (tab[s, h:] == -1).all(), s
        for b in tab[s, :h]:
            live[int(b)] = live.get(int(b), 0) + 1
    for b, c in live.items():
        assert K.kv_block_refcount(pool, b) == c
    assert K.kv_pool_stats(pool)["blocks_used"][0] == len(live)


def test_reserve_advance_share_trim_release_follow_the_model():
    pool, t = make()
    m = SeqModel(12, 40, BS)
    rng = np.random.default_rng(3)
    for step in range(400):
        op = int(rng.integers(0, 10))
        s = int(rng.integers(0, 12))
        if op < 3:
            tokens = int(rng.integers(0, 400))
            t.reserve(s, tokens)
            m.reserve(s, tokens)
        elif op < 4:
            n = int(rng.integers(0, m.held[s] * BS + 1))
            t.set_len(s, n)
            m.set_len(s, n)
        elif op < 7:
            grown_model = m.advance()
            assert t.advance() == len(grown_model)
        elif op < 8:
            t.trim(s)
            m.trim(s)
        elif op < 9:
            t.release(s)
            m.release(s)
        else:
            src = int(rng.integers(0, 12))
            if src != s and m.held[s] == 0 and m.len[s] == 0 and m.held[src] > 0:
                nb = int(rng.integers(1, m.held[src] + 1))
                t.share_prefix(s, src, nb)
                m.share_prefix(s, src, nb)
                tab, _ = t.host()
                assert np.array_equal(tab[s, :nb], tab[src, :nb])
        check_rows(t, m, pool)
    c = t.counters()
    assert c["reservation_misses"] == m.misses
    assert c["blocks_held"] == sum(m.held)
    t.close()
    assert K.kv_pool_stats(pool)["blocks_used"][0] == 0


def test_reservation_sizes_follow_eq2():
    pool, t = make()
    for tokens, blocks in [(0, 0), (1, 1), (16, 1), (17, 2), (300, 19)]:
        t.reserve(0, tokens)
        tab, _ = t.host()
        assert int((tab[0] >= 0).sum()) == blocks  # ceil(tokens / bs), never shrinking
    t.release(0)
    t.reserve(1, 33)
    assert int((t.host()[0][1] >= 0).sum()) == 3


def test_advance_is_all_or_nothing_when_the_pool_runs_out():
    pool = K.kv_pool_create(FAKE_BASE, 4 * 65536, BS, [(8, 128)], FAKE_ERR)
    t = K.SeqTab(pool, 0, 4, 8)
    for s in range(4):
        t.reserve(s, 16)
        t.set_len(s, 16)  # every slot full: the next step needs 4 new blocks, the pool has 0
    before = t.host()
    with pytest.raises(K.KVError) as e:
        t.advance()
    assert e.value.code == K.KV_ERR_OUT_OF_BLOCKS
    after = t.host()
    assert np.array_equal(before[0], after[0]) and np.array_equal(before[1], after[1])
    t.release(3)  # frees one block: one slot can now grow
    assert t.advance([0]) == 1
    with pytest.raises(K.KVError):
        t.advance([1, 1])  # duplicate slot
    t.close()


def test_shared_prefix_survives_release_of_its_origin():
    pool, t = make(S=6, max_blocks=140)
    t.reserve(0, 2048 + 100)
    t.set_len(0, 2048)
    for s in range(1, 6):
        t.share_prefix(s, 0, 128)  # 128 full blocks = a 2048-token system prompt
        t.reserve(s, 2048 + 50)
        t.set_len(s, 2048)
    tab, _ = t.host()
    prefix = tab[0, :128]
    assert all(K.kv_block_refcount(pool, int(b)) == 6 for b in prefix)
    t.release(0)
    assert all(K.kv_block_refcount(pool, int(b)) == 5 for b in prefix)
    for s in range(1, 6):
        t.release(s)
    assert K.kv_pool_stats(pool)["blocks_used"][0] == 0
    with pytest.raises(K.KVError):
        t.share_prefix(1, 2, 1)  # source holds nothing
    t.close()


def test_destroying_the_pool_first_detaches_its_tables():
    # tables closed after their pool (garbage-collection order) must not touch
    # the freed pool: they are detached and only free themselves
    pool, t = make(S=4, max_blocks=8)
    t.reserve(0, 64)
    t.set_len(0, 64)
    t2 = K.SeqTab(pool, 0, 2, 8)
    t2.reserve(1, 16)
    K.kv_pool_destroy(pool)
    for call in (lambda: t.reserve(1, 16), lambda: t.advance(), lambda: t.release(0), lambda: t2.trim(1)):
        with pytest.raises(K.KVError) as e:
            call()
        assert e.value.code == K.KV_ERR_INVALID_ARG
    t.close()
    t2.close()
    # a table destroyed before its pool unregisters itself
    pool, t = make(S=2, max_blocks=4)
    t.reserve(0, 16)
    t.close()
    assert K.kv_pool_stats(pool)["blocks_used"][0] == 0
    K.kv_pool_destroy(pool)


def test_replace_equals_release_reserve_set_len_in_order():
    """kv_seq_replace against the same operations one call at a time on a
    twin pool: identical tables (block ids included), lengths and refcounts,
    and the slot model agrees; a reservation the pool cannot serve leaves
    its slot empty while later, smaller ones are still admitted."""
    pool_a, a = make(n_pages=120)
    pool_b, b = make(n_pages=120)
    m = SeqModel(12, 40, BS)
    rng = np.random.default_rng(8)
    misses = 0
    for step in range(60):
        k = int(rng.integers(0, 7))
        slots = rng.choice(12, k, replace=False).astype(np.int32)
        res = rng.integers(0, 40 * BS + 1, size=k)
        res[rng.random(k) < 0.5] //= 8  # many small requests beside the large ones
        lens = (res * rng.random(k)).astype(np.int32)
        status = a.replace(slots, res, lens)
        for i, s in enumerate(slots):
            s = int(s)
            b.release(s)
            m.release(s)
            try:
                b.reserve(s, int(res[i]))
            except K.KVError as e:
                assert e.code == K.KV_ERR_OUT_OF_BLOCKS
                assert status[i] == K.KV_ERR_OUT_OF_BLOCKS
                misses += 1
                continue
            assert status[i] == 0
            b.set_len(s, int(lens[i]))
            m.reserve(s, int(res[i]))
            m.set_len(s, int(lens[i]))
        ta, la = a.host()
        tb, lb = b.host()
        assert np.array_equal(ta, tb) and np.array_equal(la, lb), step
        check_rows(a, m, pool_a)
        live = [s for s in range(12) if m.len[s] > 0 and m.len[s] + 1 <= m.held[s] * BS]
        if live:
            a.advance(live)
            b.advance(live)
            for s in live:
                m.len[s] += 1
    assert misses > 0  # the full-pool branch was taken
    a.close()
    b.close()


def test_replace_reports_a_full_pool_per_slot():
    pool, t = make(n_pages=8)  # 8 blocks of 16 tokens
    st = t.replace([0, 1, 2], [5 * BS, 5 * BS, 3 * BS], [10, 10, 3 * BS])
    assert list(st) == [0, K.KV_ERR_OUT_OF_BLOCKS, 0]
    _, lens = t.host()
    assert list(lens[:3]) == [10, 0, 3 * BS]
    # slot 0 replaced: its 5 blocks come back first, so slot 1's 5 now fit
    st = t.replace([0, 1], [0, 5 * BS], [0, 1])
    assert list(st) == [0, 0]
    assert K.kv_pool_stats(pool)["blocks_used"][0] == 8
    t.close()


def test_replace_checks_every_argument_before_changing_anything():
    pool, t = make()
    t.replace([0, 1], [64, 64], [10, 20])
    before = t.host()
    used = K.kv_pool_stats(pool)["blocks_used"][0]
    bad = [
        ([0, 0], [16, 16], [1, 1]),            # a slot twice
        ([0, 12], [16, 16], [1, 1]),           # slot out of range
        ([0, 1], [16, 41 * BS], [1, 1]),       # more than max_blocks
        ([0, 1], [16, -1], [1, 0]),            # negative reservation
        ([0, 1], [16, 16], [1, 17]),           # length beyond the reservation
        ([0, 1], [16, 16], [1, -1]),           # negative length
    ]
    for slots, res, lens in bad:
        with pytest.raises(K.KVError) as e:
            t.replace(slots, res, lens)
        assert e.value.code == K.KV_ERR_INVALID_ARG, (slots, res, lens)
        after = t.host()
        assert np.array_equal(before[0], after[0]) and np.array_equal(before[1], after[1])
        assert K.kv_pool_stats(pool)["blocks_used"][0] == used
    assert len(t.replace([], [], [])) == 0
    t.close()
