"""Device sync of host sequence tables: after every kv_seqtab_sync the device
table and lengths equal the host views exactly (small parameter launches,
large ones, and whole-table copies)."""
import numpy as np
import pytest

from paper_2606_12950_gb300 import kvpool as K

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _cuda():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")


@pytest.mark.parametrize("S,max_blocks", [(8, 16), (600, 40)])
def test_sync_matches_host_after_every_change(S, max_blocks):
    from paper_2606_12950_gb300.runner import DevicePool

    pool = DevicePool(S * max_blocks, 65536, 16, [(8, 128)], shuffle_seed=11)
    t = K.SeqTab(pool.handle, 0, S, max_blocks)
    dev_table = torch.full((S, max_blocks), -7, dtype=torch.int32, device="cuda")
    dev_lens = torch.full((S,), -7, dtype=torch.int32, device="cuda")
    rng = np.random.default_rng(S)
    for step in range(30):
        for _ in range(int(rng.integers(1, 40))):
            s = int(rng.integers(0, S))
            op = int(rng.integers(0, 4))
            if op == 0:
                t.reserve(s, int(rng.integers(0, max_blocks * 16 // 2)))
            elif op == 1:
                t.release(s)
            elif op == 2:
                tab, lens = t.host()
                t.set_len(s, int(rng.integers(0, (tab[s] >= 0).sum() * 16 + 1)))
            else:
                t.trim(s)
        tab, lens = t.host()
        live = [s for s in range(S) if 0 < lens[s] < max_blocks * 16 - 1]
        if live:
            t.advance(live)
        if step == 17:  # touch most of the table: whole-table copy path
            for s in range(S):
                t.release(s)
                t.reserve(s, 16 * (max_blocks // 2))
        t.sync(dev_table, dev_lens)
        torch.cuda.synchronize()
        tab, lens = t.host()
        assert np.array_equal(dev_table.cpu().numpy(), tab), step
        assert np.array_equal(dev_lens.cpu().numpy(), lens), step
    c = t.counters()
    assert c["sync_launches"] >= 30
    t.close()
    pool.close()


@pytest.mark.parametrize("S", [24, 300])
def test_fused_sync_gives_the_bits_of_sync_then_attention(S):
    """paged_decode_attn_seqtab against kv_seqtab_sync followed by
    paged_decode_attn_append, on two pools with the same contents driven by
    the same table operations: after every step the outputs, the pools (with
    the appended rows), the device tables and the lengths are bit-identical.
    The steps cover launches that carry the sync (few changes), the separate
    sync kernel (many changes, or more rows than the parameters hold) and the
    first whole-table copy."""
    from paper_2606_12950_gb300.runner import DevicePool, DeviceSteps

    Hq, Hkv, d, bs, max_blocks = 8, 2, 128, 16, 12
    n_pages = S * max_blocks + 8
    page_elems = 2 * Hkv * bs * d
    rng = np.random.default_rng(77)
    host_pool = (rng.standard_normal(n_pages * page_elems).astype(np.float32).view(np.uint32) >> 16).astype(np.uint16)
    q = (rng.standard_normal((S, Hq, d)).astype(np.float32).view(np.uint32) >> 16).astype(np.uint16)
    kn = (rng.standard_normal((S, Hkv, d)).astype(np.float32).view(np.uint32) >> 16).astype(np.uint16)
    vn = (rng.standard_normal((S, Hkv, d)).astype(np.float32).view(np.uint32) >> 16).astype(np.uint16)
    sides = []
    for _ in range(2):
        pool = DevicePool(n_pages, page_elems * 2, bs, [(Hkv, d)], shuffle_seed=3)
        pool.upload(host_pool)
        t = K.SeqTab(pool.handle, 0, S, max_blocks)
        buf = DeviceSteps(pool, 0, S, S, Hq, Hkv, d, max_blocks, d ** -0.5, q, kn, vn)
        sides.append((pool, t, buf))
    ops = np.random.default_rng(S)
    for s in range(S):
        tokens = int(ops.integers(1, 6 * bs))
        for _, t, _ in sides:
            t.reserve(s, tokens + 2 * bs)
            t.set_len(s, tokens)
    for step in range(12):
        if step == 6:  # many changes at once: the separate sync kernel
            for s in range(0, S, 2):
                for _, t, _ in sides:
                    t.release(s)
                    t.reserve(s, 3 * bs)
                    t.set_len(s, 2 * bs - 1)
        for _, t, _ in sides:
            tab, lens = t.host()
            t.advance([s for s in range(S) if lens[s] + 1 < max_blocks * bs])
        pool_a, t_a, buf_a = sides[0]
        t_a.sync(buf_a.table, buf_a.lens)
        buf_a.append_attend()
        pool_b, t_b, buf_b = sides[1]
        buf_b.sync_append_attend(t_b)
        torch.cuda.synchronize()
        assert np.array_equal(buf_a.out.cpu().view(torch.int16).numpy(), buf_b.out.cpu().view(torch.int16).numpy()), step
        assert np.array_equal(buf_a.table.cpu().numpy(), buf_b.table.cpu().numpy()), step
        assert np.array_equal(buf_a.lens.cpu().numpy(), buf_b.lens.cpu().numpy()), step
        assert np.array_equal(pool_a.download(), pool_b.download()), step
        tab, lens = t_b.host()
        assert np.array_equal(buf_b.table.cpu().numpy(), tab) and np.array_equal(buf_b.lens.cpu().numpy(), lens)
        assert pool_a.error() == 0 and pool_b.error() == 0
    for pool, t, _ in sides:
        t.close()
        pool.close()
