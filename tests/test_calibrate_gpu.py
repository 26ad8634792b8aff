"""The decode-latency microbenchmark on the GPU: a small grid of one layer
shape, checked for the structure Eq. 1's t_dec relies on (time grows with
the KV streamed; the linear cost model fits)."""
import pytest

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _cuda():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")


def test_small_calibration_grid():
    from paper_2606_12950_gb300 import calibrate as C

    res = C.calibrate({"gqa-32x8-d128": (32, 8, 128)}, batches=(1, 8, 32), contexts=(512, 4096), iters=8)
    r = res["gqa-32x8-d128"]
    t = {(s["B"], s["n"]): s["seconds"] for s in r["samples"]}
    assert t[(32, 4096)] > t[(32, 512)] and t[(32, 4096)] > t[(8, 4096)]
    assert r["r2"] > 0.9
    assert r["effective_gbs"] is not None and r["effective_gbs"] > 500  # bandwidth-bound at scale
    assert all(s["seconds"] > 0 for s in r["samples"])
