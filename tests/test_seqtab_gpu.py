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
