"""The allocation-free attention entry point (paged_decode_attn_noalloc).

Some callers cannot allocate device memory when they run attention: their KV
pool already holds all free HBM, their framework owns the allocator, or a
cudaMalloc (which may synchronise the device) is not acceptable inside the
decode loop.  paged_decode_attn_noalloc uses a fixed scratch array inside the
library instead of a caller workspace.  These tests call it through the C
ABI, twice in a row, and check each result against the fp64 oracle and
against paged_decode_attn with a caller workspace, within the parity
tolerance of the other GPU tests: with automatic and with forced split
counts (so the scratch holds split partials), after a call of a larger
shape (so the scratch holds another call's leftovers), and, in a fresh
process, with the first call made only after the pool was created (the
scratch was taken at pool creation, so the first call takes no device
memory).  The file is named so pytest collects it last.
"""
import os
import subprocess
import sys

import numpy as np
import pytest

import oracle
from paper_2606_12950_gb300 import workloads as W

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

MAX_ABS = 1.5e-2
MEAN_ABS = 2e-3
SCRATCH_BYTES = 32 << 20
ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module", autouse=True)
def _cuda():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")


def _close(a, b):
    err = np.abs(a - b)
    assert np.isfinite(a).all()
    assert err.max() <= MAX_ABS and err.mean() <= MEAN_ABS, (err.max(), err.mean())


def _setup(b):
    from paper_2606_12950_gb300.runner import DeviceBatch, DevicePool

    pool = DevicePool(b.n_pages, b.page_elems * 2, b.bs, [(b.Hkv, b.d)])
    pool.upload(b.pool)
    db = DeviceBatch(pool, 0, b)
    db.append()
    torch.cuda.synchronize()
    return pool, db


def _noalloc(pool, db, b, num_splits):
    from paper_2606_12950_gb300 import kvpool as K

    out = torch.full_like(db.out, float("nan"))
    K.paged_decode_attn_noalloc(pool.handle, 0, db.q, out, db.table, db.lens, b.max_blocks, b.S, b.Hq, b.scale,
                                num_splits, torch.cuda.current_stream())
    torch.cuda.synchronize()
    return out.float().cpu().numpy().astype(np.float64)


@pytest.mark.parametrize("which", ["tiny", "llama8b"])
@pytest.mark.parametrize("num_splits", [0, 5])
def test_noalloc_matches_oracle_and_workspace_path_twice(which, num_splits):
    b = W.config1_tiny() if which == "tiny" else W.config2_llama8b()
    pool, db = _setup(b)
    ref_pool = oracle.batch_append(b)
    ref = oracle.batch_attention(b, pool=ref_pool)
    db.attend(num_splits=num_splits)
    torch.cuda.synchronize()
    ws_out = db.out_f64()
    _close(ws_out, ref)
    for call in range(2):
        got = _noalloc(pool, db, b, num_splits)
        _close(got, ref)
        _close(got, ws_out)
    assert pool.error() == 0
    pool.close()


def test_noalloc_after_a_larger_call_leaves_no_trace():
    """A call with many splits of the full-size batch fills the scratch with
    its partials; a following call on the small batch (fewer runs, other
    splits) must not read them: it matches its workspace result and the
    oracle, twice."""
    big = W.config2_llama8b()
    pool_b, db_b = _setup(big)
    _noalloc(pool_b, db_b, big, 64)
    small = W.config1_tiny()
    pool_s, db_s = _setup(small)
    ref = oracle.batch_attention(small, pool=oracle.batch_append(small))
    for ns in (3, 0):
        db_s.attend(num_splits=ns)
        torch.cuda.synchronize()
        ws_out = db_s.out_f64()
        for call in range(2):
            got = _noalloc(pool_s, db_s, small, ns)
            _close(got, ws_out)
            _close(got, ref)
    assert pool_b.error() == 0 and pool_s.error() == 0
    pool_b.close()
    pool_s.close()


_FRESH = r"""
import sys
sys.path.insert(0, sys.argv[1])
import numpy as np, torch
import oracle
from paper_2606_12950_gb300 import kvpool as K, workloads as W
from paper_2606_12950_gb300.runner import DeviceBatch, DevicePool
torch.cuda.set_device(0)
b = W.config1_tiny()
pool = DevicePool(b.n_pages, b.page_elems * 2, b.bs, [(b.Hkv, b.d)])
pool.upload(b.pool)
db = DeviceBatch(pool, 0, b)
db.append()
db.attend(num_splits=3)     # loads the attention kernels' modules
torch.cuda.synchronize()
free0 = torch.cuda.mem_get_info()[0]
out = torch.full_like(db.out, float("nan"))
K.paged_decode_attn_noalloc(pool.handle, 0, db.q, out, db.table, db.lens, b.max_blocks, b.S, b.Hq, b.scale, 3,
                            torch.cuda.current_stream())
torch.cuda.synchronize()
free1 = torch.cuda.mem_get_info()[0]
ref = oracle.batch_attention(b, pool=oracle.batch_append(b))
err = np.abs(out.float().cpu().numpy().astype(np.float64) - ref)
print("RESULT", free0 - free1, err.max(), err.mean(), pool.error())
"""


def test_first_call_after_pool_creation_takes_no_device_memory():
    """In a fresh process: create a pool (which takes the scratch on the
    device), run the workspace path once, then make the first noalloc call.
    The device's free memory must not drop by the scratch's 32 MiB at that
    call, and the result matches the oracle."""
    r = subprocess.run([sys.executable, "-c", _FRESH, ROOT], capture_output=True, text=True, timeout=600)
    assert r.returncode == 0, r.stderr[-3000:]
    line = [l for l in r.stdout.splitlines() if l.startswith("RESULT")][-1].split()
    drop, emax, emean, err = int(line[1]), float(line[2]), float(line[3]), int(line[4])
    assert drop < SCRATCH_BYTES, drop
    assert emax <= MAX_ABS and emean <= MEAN_ABS and err == 0


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
