"""The VMM-backed elastic pool on the GPU (CUDA virtual memory backend):
decode parity of the fused append + attention over blocks the allocator
mapped on demand, device memory that follows allocation and trim, and
several pools whose reserved virtual KV far exceeds a shared physical budget
(the overcommitment of §III-C / Table 5)."""
import numpy as np
import pytest

import oracle
from paper_2606_12950_gb300 import kvpool as K
from paper_2606_12950_gb300 import workloads as W

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

GB = 1 << 30
MB = 1 << 20
BLOCK = 2 * 8 * 16 * 128 * 2  # 8 KV heads, bs 16, d 128


@pytest.fixture(scope="module", autouse=True)
def _cuda():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")


def test_decode_parity_on_blocks_mapped_on_demand():
    from paper_2606_12950_gb300.runner import DeviceBatch, VmmPool

    b = W.make_batch(7001, [17, 300, 1023, 2500, 64, 5, 900, 4000], Hq=32, Hkv=8, d=128, bs=16)
    pool = VmmPool(8 * GB, BLOCK, 16, [(8, 128)], physical_limit=1 * GB, shuffle_seed=3)
    assert pool.stats()["bytes_mapped"] == 0
    ids = K.kv_alloc_blocks(pool.handle, 0, b.n_pages)  # compact id i lives at VMM block ids[i]
    assert 0 < pool.stats()["bytes_mapped"] <= 1 * GB
    pool.write_pages(ids, b.pool.reshape(b.n_pages, b.page_elems))
    vb = W.Batch(**{**b.__dict__})
    vb.table = np.where(b.table >= 0, ids[np.maximum(b.table, 0)], -1).astype(np.int32)
    db = DeviceBatch(pool, 0, vb)
    db.append_attend()
    torch.cuda.synchronize()
    ref_pool = oracle.batch_append(b)
    assert np.array_equal(pool.read_pages(ids), ref_pool.reshape(b.n_pages, b.page_elems))
    err = np.abs(db.out_f64() - oracle.batch_attention(b, pool=ref_pool))
    assert err.max() <= 1.5e-2 and err.mean() <= 2e-3, (err.max(), err.mean())
    assert pool.error() == 0
    pool.close()


def test_device_memory_follows_allocation_and_trim():
    from paper_2606_12950_gb300.runner import VmmPool

    torch.cuda.synchronize()
    pool = VmmPool(16 * GB, BLOCK, 16, [(8, 128)])
    free0 = torch.cuda.mem_get_info()[0]
    n = (2 * GB) // BLOCK
    ids = K.kv_alloc_blocks(pool.handle, 0, n)
    mapped = pool.stats()["bytes_mapped"]
    assert mapped >= 2 * GB
    free1 = torch.cuda.mem_get_info()[0]
    assert free0 - free1 >= 2 * GB - 64 * MB
    pool.fill_random(ids[:64], 5)  # the mapped blocks are usable memory
    K.kv_free_blocks(pool.handle, 0, ids)
    assert pool.stats()["bytes_mapped"] == mapped  # freed blocks stay mapped until trim
    released = pool.trim()
    assert released == mapped and pool.stats()["bytes_mapped"] == 0
    free2 = torch.cuda.mem_get_info()[0]
    assert abs(free2 - free0) <= 64 * MB
    pool.close()


def test_overcommitted_pools_share_a_physical_budget():
    """Three pools reserve 16 GB of virtual KV each (48 GB) over a 2 GB
    budget (24x): allocation succeeds up to the budget, is then rejected
    whole, and one pool's trim lets another grow."""
    from paper_2606_12950_gb300.runner import VmmPool

    bud = K.kv_budget_create(2 * GB)
    pools = [VmmPool(16 * GB, BLOCK, 16, [(8, 128)], budget=bud, shuffle_seed=i + 1) for i in range(3)]
    a = K.kv_alloc_blocks(pools[0].handle, 0, (1 * GB) // BLOCK)
    K.kv_alloc_blocks(pools[1].handle, 0, (1 * GB) // BLOCK)
    assert K.kv_budget_used(bud) == 2 * GB
    with pytest.raises(K.KVError) as e:
        K.kv_alloc_blocks(pools[2].handle, 0, 1)
    assert e.value.code == K.KV_ERR_OUT_OF_BLOCKS
    assert pools[2].stats()["blocks_used"][0] == 0
    K.kv_free_blocks(pools[0].handle, 0, a)
    assert pools[0].trim() == 1 * GB
    c = K.kv_alloc_blocks(pools[2].handle, 0, (1 * GB) // BLOCK)
    pools[2].fill_random(c[-16:], 9)
    assert K.kv_budget_used(bud) == 2 * GB
    for p in pools:
        p.close()
    assert K.kv_budget_used(bud) == 0
    K.kv_budget_destroy(bud)


def test_table_upload_refuses_unmapped_blocks():
    from paper_2606_12950_gb300.runner import VmmPool

    pool = VmmPool(4 * GB, BLOCK, 16, [(8, 128)])
    ids = K.kv_alloc_blocks(pool.handle, 0, 4)
    table = torch.full((1, 8), -1, dtype=torch.int32, device="cuda")
    lens = torch.zeros(1, dtype=torch.int32, device="cuda")
    host = np.full((1, 8), -1, np.int32)
    host[0, :4] = ids
    K.kv_block_table_upload(pool.handle, 0, host, np.array([64], np.int32), table, lens)
    far = pool.n_pages - 1  # in the reserved range, never mapped
    host[0, 3] = far
    with pytest.raises(K.KVError) as e:
        K.kv_block_table_upload(pool.handle, 0, host, np.array([64], np.int32), table, lens)
    assert e.value.code == K.KV_ERR_INVALID_ARG
    torch.cuda.synchronize()
    pool.close()
