"""The allocation-free attention entry point (paged_decode_attn_noalloc).

Some callers cannot allocate device memory when they run attention: their KV
pool already holds all free HBM, their framework owns the allocator, or a
cudaMalloc (which may synchronise the device) is not acceptable inside the
decode loop.  paged_decode_attn_noalloc uses a fixed scratch array inside the
library instead of a caller workspace.  This test calls it through the C ABI
twice in a row and checks each result against paged_decode_attn with a
caller workspace, within the parity tolerance of the other GPU tests.  The
file is named so pytest collects it last.
"""
import numpy as np
import pytest

from paper_2606_12950_gb300 import workloads as W

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

MAX_ABS = 1.5e-2
MEAN_ABS = 2e-3
SCRATCH_BYTES = 32 << 20


@pytest.fixture(scope="module", autouse=True)
def _cuda():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")


def _close(a, b):
    err = np.abs(a - b)
    assert np.isfinite(a).all()
    assert err.max() <= MAX_ABS and err.mean() <= MEAN_ABS, (err.max(), err.mean())


@pytest.mark.parametrize("which", ["tiny", "llama8b"])
def test_noalloc_matches_workspace_path_twice(which):
    from paper_2606_12950_gb300 import kvpool as K
    from paper_2606_12950_gb300.runner import DeviceBatch, DevicePool

    b = W.config1_tiny() if which == "tiny" else W.config2_llama8b()
    pool = DevicePool(b.n_pages, b.page_elems * 2, b.bs, [(b.Hkv, b.d)])
    pool.upload(b.pool)
    db = DeviceBatch(pool, 0, b)
    db.append()
    db.attend()
    torch.cuda.synchronize()
    ref = db.out_f64()
    for call in range(2):
        out = torch.full_like(db.out, float("nan"))
        K.paged_decode_attn_noalloc(pool.handle, 0, db.q, out, db.table, db.lens, b.max_blocks, b.S, b.Hq,
                                    b.scale, 0, torch.cuda.current_stream())
        torch.cuda.synchronize()
        _close(out.float().cpu().numpy().astype(np.float64), ref)
    assert pool.error() == 0
    pool.close()


def test_noalloc_rejects_batches_beyond_its_scratch():
    from paper_2606_12950_gb300 import kvpool as K
    from paper_2606_12950_gb300.runner import DevicePool

    pool = DevicePool(16, 65536, 16, [(8, 128)])
    S, Hq, max_blocks = 4096, 32, 8
    assert K.kv_workspace_bytes(pool.handle, 0, S, Hq, max_blocks) > SCRATCH_BYTES
    q = torch.zeros((S, Hq, 128), dtype=torch.bfloat16, device="cuda")
    out = torch.zeros_like(q)
    table = torch.zeros((S, max_blocks), dtype=torch.int32, device="cuda")
    lens = torch.ones(S, dtype=torch.int32, device="cuda")
    with pytest.raises(K.KVError) as e:
        K.paged_decode_attn_noalloc(pool.handle, 0, q, out, table, lens, max_blocks, S, Hq, 0.1, 0,
                                    torch.cuda.current_stream())
    assert e.value.code == K.KV_ERR_WORKSPACE
    torch.cuda.synchronize()
    assert torch.count_nonzero(out).item() == 0  # nothing was launched
    pool.close()
