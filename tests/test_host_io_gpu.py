"""Host buffers through the C ABI: q, k_new, v_new and out may be pinned
(mapped) host memory, which the kernels read and write directly over the
GPU's coherent link to host memory.  The results must be the bits that the
same calls give with device buffers: the pool after the fused append, the
attention output, the shared-prefix (cascade) output and the output of
several batches in one paged_decode_attn_multi call."""
import numpy as np
import pytest

from paper_2606_12950_gb300 import kvpool as K
from paper_2606_12950_gb300 import workloads as W

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _cuda():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")


def _pinned_like(t, fill=None):
    h = torch.empty(t.shape, dtype=t.dtype).pin_memory()
    if fill is None:
        h.copy_(t.cpu())
    else:
        h.fill_(fill)
    return h


def _run(b, host: bool, call):
    from paper_2606_12950_gb300.runner import DeviceBatch, DevicePool

    pool = DevicePool(b.n_pages, b.page_elems * 2, b.bs, [(b.Hkv, b.d)])
    pool.upload(b.pool)
    db = DeviceBatch(pool, 0, b)
    if host:
        db.q, db.k_new, db.v_new = (_pinned_like(t) for t in (db.q, db.k_new, db.v_new))
        db.out = _pinned_like(db.out, float("nan"))
    call(db)
    torch.cuda.synchronize()
    out = db.out.cpu().view(torch.int16).numpy().copy()
    res = (out, pool.download(), pool.error())
    pool.close()
    return res


@pytest.mark.parametrize("which", ["tiny", "llama8b"])
@pytest.mark.parametrize("fused", [True, False], ids=["fused", "separate"])
def test_host_buffers_give_the_device_bits(which, fused):
    b = W.config1_tiny() if which == "tiny" else W.config2_llama8b()

    def call(db):
        if fused:
            db.append_attend()
        else:
            db.append()
            db.attend()

    dev = _run(b, False, call)
    host = _run(b, True, call)
    assert dev[2] == 0 and host[2] == 0
    assert np.array_equal(dev[0], host[0]), "attention output differs with host buffers"
    assert np.array_equal(dev[1], host[1]), "pool after the append differs with host buffers"


def test_host_buffers_shared_prefix():
    b = W.make_batch(77, [300, 290, 400, 280, 700, 350], Hq=32, Hkv=8, d=128, bs=16, extra_blocks=4)
    groups = [(range(0, 6), 256)]
    W.share_prefix(b, groups)

    def call(db):
        db.cascade(K.PrefixPlan(groups), fused=True)

    dev = _run(b, False, call)
    host = _run(b, True, call)
    assert dev[2] == 0 and host[2] == 0
    assert np.array_equal(dev[0], host[0]), "cascade output differs with host buffers"
    assert np.array_equal(dev[1], host[1]), "pool after the append differs with host buffers"


def test_host_buffers_multi_batch():
    """paged_decode_attn_multi (a chain of decode kernels) over two halves of
    one batch, with the fused append: host q, new rows and out give the
    device-buffer bits (outputs and pool)."""
    from paper_2606_12950_gb300.runner import DeviceBatch, DevicePool

    b = W.make_batch(81, [40, 900, 333, 1200, 5, 77, 2048, 610], Hq=32, Hkv=8, d=128, bs=16, extra_blocks=4)
    h = b.S // 2

    def run(host: bool):
        pool = DevicePool(b.n_pages, b.page_elems * 2, b.bs, [(b.Hkv, b.d)])
        pool.upload(b.pool)
        db = DeviceBatch(pool, 0, b)
        if host:
            db.q, db.k_new, db.v_new = (_pinned_like(t) for t in (db.q, db.k_new, db.v_new))
            db.out = _pinned_like(db.out, float("nan"))
        entries = []
        for lo, hi in ((0, h), (h, b.S)):
            need = K.kv_workspace_bytes(pool.handle, 0, hi - lo, b.Hq, b.max_blocks)
            ws = torch.zeros(need, dtype=torch.uint8, device="cuda")
            entries.append(dict(db.batch(), q=db.q[lo:hi], k_new=db.k_new[lo:hi], v_new=db.v_new[lo:hi],
                                out=db.out[lo:hi], dev_table=db.table[lo:hi], dev_ctx_lens=db.lens[lo:hi],
                                S=hi - lo, workspace=ws, ws_bytes=need))
        K.paged_decode_attn_multi(pool.handle, entries)
        torch.cuda.synchronize()
        res = (db.out.cpu().view(torch.int16).numpy().copy(), pool.download(), pool.error())
        pool.close()
        return res

    dev, host = run(False), run(True)
    assert dev[2] == 0 and host[2] == 0
    assert np.array_equal(dev[0], host[0]), "multi-batch output differs with host buffers"
    assert np.array_equal(dev[1], host[1]), "pool after the append differs with host buffers"
