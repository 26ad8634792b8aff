"""CPU-only checks of the C ABI: the library loads and exports every entry
point the header declares; the host-side pool allocator against the
accounting model in oracle/alloc_model.py; argument validation that happens
before anything is launched.  No kernel runs here."""
import os
import re

import numpy as np
import pytest

from oracle.alloc_model import AllocModel
from paper_2606_12950_gb300 import kvpool as K

HEADER = os.path.join(os.path.dirname(os.path.dirname(os.path.abspath(__file__))), "include", "kvpool.h")
FAKE_BASE = 1 << 40  # host-only tests never dereference the device pointer
FAKE_ERR = (1 << 40) + (1 << 30)


def declared_functions():
    text = open(HEADER).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"^\s*(?:int|const char \*)\s*\**\s*([a-z_]+)\s*\(", text, flags=re.M)))


def test_library_exports_every_declared_entry_point():
    L = K.lib()
    names = declared_functions()
    assert len(names) >= 15
    for n in names:
        assert hasattr(L, n), n
    assert "sm_103a" in K.kv_version()


def make_pool(n_pages=64, layouts=((8, 128),), bs=16, page_bytes=0, seed=0):
    block = min(2 * h * bs * d * 2 for h, d in layouts)
    pb = page_bytes or block
    return K.kv_pool_create(FAKE_BASE, n_pages * pb, bs, list(layouts), FAKE_ERR, page_bytes=pb,
                            shuffle_seed=seed), pb


def test_create_rejects_bad_descriptors():
    with pytest.raises(K.KVError):
        K.kv_pool_create(FAKE_BASE + 8, 1 << 20, 16, [(8, 128)], FAKE_ERR)  # misaligned base
    with pytest.raises(K.KVError):
        K.kv_pool_create(FAKE_BASE, 1 << 20, 0, [(8, 128)], FAKE_ERR)  # bs = 0
    with pytest.raises(K.KVError):
        K.kv_pool_create(FAKE_BASE, 1 << 20, 16, [], FAKE_ERR)
    with pytest.raises(K.KVError):
        K.kv_pool_create(FAKE_BASE, 1 << 10, 16, [(8, 128)], FAKE_ERR)  # smaller than one block
    with pytest.raises(K.KVError):  # 65536-byte and 98304-byte blocks cannot share a page size
        K.kv_pool_create(FAKE_BASE, 1 << 24, 16, [(8, 128), (12, 128)], FAKE_ERR)


@pytest.mark.parametrize("seed", [0, 7])
def test_allocator_matches_accounting_model(seed):
    layouts = [(32, 128), (8, 128), (8, 128)]  # 256 KiB and 64 KiB blocks, 64 KiB pages
    h, pb = make_pool(n_pages=4 * 40 + 3, layouts=layouts, seed=seed)
    model = AllocModel(4 * 40 + 3, [4, 1, 1])
    rng = np.random.default_rng(seed + 100)
    live = {0: [], 1: [], 2: []}
    for step in range(600):
        op = rng.integers(0, 10)
        lay = int(rng.integers(0, 3))
        if op < 5:
            n = int(rng.integers(0, 12))
            try:
                ids = K.kv_alloc_blocks(h, lay, n)
                assert model.alloc(lay, n, [int(i) for i in ids]), (step, lay, n)
                live[lay].extend(int(i) for i in ids)
            except K.KVError as e:
                assert e.code == K.KV_ERR_OUT_OF_BLOCKS
                assert model.alloc(lay, n, None), (step, lay, n)
        elif op < 8 and live[lay]:
            k = int(rng.integers(1, min(6, len(live[lay])) + 1))
            pick = [live[lay].pop(int(rng.integers(0, len(live[lay])))) for _ in range(k)]
            assert model.free_ok(lay, pick)
            K.kv_free_blocks(h, lay, pick)
            model.free(lay, pick)
        elif live[lay]:
            pick = [live[lay][int(rng.integers(0, len(live[lay])))]]
            K.kv_block_ref(h, lay, pick)
            model.add_ref(pick)
            live[lay].extend(pick)
        st = K.kv_pool_stats(h)
        for l in range(3):
            assert st["blocks_used"][l] == model.used(l)
            assert st["blocks_capacity"][l] == model.used(l) + model.capacity(l)
        for i, c in list(model.ref.items())[:5]:
            assert K.kv_block_refcount(h, i) == c
    # blocks of one layout never overlap blocks of another
    spans = []
    for l, ids in live.items():
        k = [4, 1, 1][l]
        spans += [(i, i + k) for i in set(ids)]
    spans.sort()
    for (a0, a1), (b0, b1) in zip(spans, spans[1:]):
        assert a1 <= b0
    K.kv_pool_destroy(h)


def test_free_and_ref_validation_changes_nothing():
    h, _ = make_pool(n_pages=16)
    ids = K.kv_alloc_blocks(h, 0, 4)
    before = K.kv_pool_stats(h)
    with pytest.raises(K.KVError):
        K.kv_free_blocks(h, 0, [ids[0], ids[0]])  # two drops of a block holding one reference
    with pytest.raises(K.KVError):
        K.kv_free_blocks(h, 0, [ids[1], 15 if 15 not in ids else 14])  # second id not live
    with pytest.raises(K.KVError):
        K.kv_block_ref(h, 0, [-1])
    assert K.kv_pool_stats(h) == before
    K.kv_block_ref(h, 0, [ids[0]])
    K.kv_free_blocks(h, 0, [ids[0], ids[0]])  # now it holds two
    assert K.kv_block_refcount(h, int(ids[0])) == 0
    with pytest.raises(K.KVError):
        K.kv_alloc_blocks(h, 0, 14)  # 13 free
    assert K.kv_pool_stats(h)["blocks_used"][0] == 3
    K.kv_pool_destroy(h)


def test_stats_of_a_fresh_pool():
    """kv_stats as the binding reads it: a fresh pool's pages, bytes and its
    count of overlapped attention calls (the last field: a layout mismatch
    between the header and the binding shows here)."""
    h, _ = make_pool(n_pages=16)
    st = K.kv_pool_stats(h)
    assert st["pages_total"] == 16
    assert st["bytes_used"] == 0 and st["bytes_mapped"] == st["bytes_total"] > 0
    assert st["attn_calls_overlapped"] == 0
    K.kv_set_attn_step_overlap(h, 1)
    assert K.kv_pool_stats(h)["attn_calls_overlapped"] == 0
    K.kv_pool_destroy(h)


def test_shuffled_free_order_is_a_seeded_permutation():
    h1, _ = make_pool(n_pages=256, seed=42)
    h2, _ = make_pool(n_pages=256, seed=42)
    h3, _ = make_pool(n_pages=256, seed=0)
    a = K.kv_alloc_blocks(h1, 0, 256)
    b = K.kv_alloc_blocks(h2, 0, 256)
    c = K.kv_alloc_blocks(h3, 0, 256)
    assert np.array_equal(a, b)
    assert sorted(a.tolist()) == list(range(256))
    assert c.tolist() == list(range(256))
    assert a.tolist() != c.tolist()


def test_table_upload_validates_on_host_before_copying():
    h, _ = make_pool(n_pages=16)
    table = np.zeros((2, 4), np.int32)
    # length beyond max_blocks * bs
    with pytest.raises(K.KVError) as e:
        K.kv_block_table_upload(h, 0, table, [10, 65], 1 << 40, 1 << 40)
    assert e.value.code == K.KV_ERR_INVALID_ARG
    # reachable entry outside the pool
    table[1, 1] = 16
    with pytest.raises(K.KVError):
        K.kv_block_table_upload(h, 0, table, [10, 17], 1 << 40, 1 << 40)
    # negative length
    with pytest.raises(K.KVError):
        K.kv_block_table_upload(h, 0, table, [-1, 3], 1 << 40, 1 << 40)


def test_attention_argument_checks_precede_any_launch():
    h, _ = make_pool(n_pages=16)
    with pytest.raises(K.KVError) as e:  # Hq not a multiple of Hkv
        K.kv_workspace_bytes(h, 0, 4, 12, 8)
    assert e.value.code == K.KV_ERR_INVALID_ARG
    with pytest.raises(K.KVError) as e:  # G = 3 is not built
        K.kv_workspace_bytes(h, 0, 4, 24, 8)
    assert e.value.code == K.KV_ERR_UNSUPPORTED
    with pytest.raises(K.KVError) as e:
        K.paged_decode_attn(h, 1, 0, 0, 0, 0, 8, 4, 32, 0.1, 0, 0, 0)  # no layout 1
    assert e.value.code == K.KV_ERR_INVALID_ARG
    h2 = K.kv_pool_create(FAKE_BASE, 64 * 49152, 16, [(12, 64)], FAKE_ERR)
    with pytest.raises(K.KVError) as e:  # d = 64 fine, G = 1 fine, but d=96 is not
        K.kv_pool_create(FAKE_BASE, 64 * 49152, 16, [(8, 96)], FAKE_ERR) and None
        K.kv_workspace_bytes(K.kv_pool_create(FAKE_BASE, 1 << 26, 16, [(8, 96)], FAKE_ERR), 0, 1, 8, 1)
    assert e.value.code == K.KV_ERR_UNSUPPORTED
    K.kv_pool_destroy(h2)
    # S = 0 is a no-op that needs no buffers
    K.paged_decode_attn(h, 0, 0, 0, 0, 0, 8, 0, 32, 0.1, 0, 0, 0)
    K.kv_append(h, 0, 0, 0, 0, 0, 8, 0)


def test_multi_batch_checks_every_batch_before_launching():
    h, _ = make_pool(n_pages=16)
    empty = dict(layout=0, q=0, out=0, dev_table=0, dev_ctx_lens=0, max_blocks=8, S=0, Hq=32, scale=0.1,
                 workspace=0, ws_bytes=0)
    K.paged_decode_attn_multi(h, [])               # nothing to do
    K.paged_decode_attn_multi(h, [empty, empty])   # S = 0 batches are skipped: nothing is launched
    for bad, code in [(dict(empty, S=4, Hq=12), K.KV_ERR_INVALID_ARG),   # Hq not a multiple of Hkv
                      (dict(empty, S=4, Hq=24), K.KV_ERR_UNSUPPORTED),   # G = 3 is not built
                      (dict(empty, S=4), K.KV_ERR_INVALID_ARG),          # no q / out / table
                      (dict(empty, layout=1), K.KV_ERR_INVALID_ARG),     # no layout 1
                      (dict(empty, scale=float("nan")), K.KV_ERR_INVALID_ARG)]:
        with pytest.raises(K.KVError) as e:  # a bad batch after a good one: the call launches nothing
            K.paged_decode_attn_multi(h, [empty, bad])
        assert e.value.code == code, bad
    assert K.lib().paged_decode_attn_multi(h, -1, None, None) == K.KV_ERR_INVALID_ARG


def test_seqtab_attention_argument_checks_precede_any_launch():
    h, _ = make_pool(n_pages=16)
    h2, _ = make_pool(n_pages=16)
    t = K.SeqTab(h, 0, 4, 8)
    fake = 1 << 41  # never dereferenced: every call below fails its host checks
    cases = [
        (h2, t, dict(S=4), K.KV_ERR_INVALID_ARG),                  # table over another pool
        (h, t, dict(S=5), K.KV_ERR_INVALID_ARG),                   # more rows than the table has
        (h, t, dict(S=4, dev_table=None), K.KV_ERR_INVALID_ARG),   # no device table
        (h, t, dict(S=4, v_new=None), K.KV_ERR_INVALID_ARG),       # k_new without v_new
    ]
    for pool, tab, over, code in cases:
        args = dict(q=fake, k_new=fake, v_new=fake, out=fake, dev_table=fake, dev_lens=fake, S=4)
        args.update(over)
        with pytest.raises(K.KVError) as e:
            K.paged_decode_attn_seqtab(pool, tab, args["q"], args["k_new"], args["v_new"], args["out"],
                                       args["dev_table"], args["dev_lens"], args["S"], 32, 0.1, 0, fake, 1 << 20)
        assert e.value.code == code, over
    t.close()


def test_cascade_seqtab_argument_checks_precede_any_launch():
    h, _ = make_pool(n_pages=16)
    h2, _ = make_pool(n_pages=16)
    t = K.SeqTab(h, 0, 4, 8)
    fake = 1 << 41  # never dereferenced: every call below fails its host checks
    plan = K.PrefixPlan([([0, 1], 64)])
    cases = [
        (h2, t, dict(S=4), K.KV_ERR_INVALID_ARG),                  # table over another pool
        (h, t, dict(S=5), K.KV_ERR_INVALID_ARG),                   # more rows than the table has
        (h, t, dict(S=4, dev_table=None), K.KV_ERR_INVALID_ARG),   # no device table
        (h, t, dict(S=4, v_new=None), K.KV_ERR_INVALID_ARG),       # k_new without v_new
    ]
    for pool, tab, over, code in cases:
        args = dict(q=fake, k_new=fake, v_new=fake, out=fake, dev_table=fake, dev_lens=fake, S=4)
        args.update(over)
        with pytest.raises(K.KVError) as e:
            K.paged_decode_attn_cascade_seqtab(pool, tab, args["q"], args["k_new"], args["v_new"], args["out"],
                                               args["dev_table"], args["dev_lens"], args["S"], 32, 0.1, plan,
                                               fake, 1 << 20)
        assert e.value.code == code, over
    rc = K.lib().paged_decode_attn_cascade_seqtab(h, t.handle, fake, fake, fake, fake, fake, fake, 4, 32,
                                                  0.1, None, -1, None, fake, 1 << 20, None)
    assert rc == K.KV_ERR_INVALID_ARG  # a negative group count
    t.close()


def test_step_overlap_switch_checks_its_arguments():
    h, _ = make_pool(n_pages=16)
    K.kv_set_attn_step_overlap(h, True)
    K.kv_set_attn_step_overlap(h, False)
    assert K.lib().kv_set_attn_step_overlap(h, 2) == K.KV_ERR_INVALID_ARG
    assert K.lib().kv_set_attn_step_overlap(None, 1) == K.KV_ERR_INVALID_ARG
