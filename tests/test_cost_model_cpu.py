"""Eq. 1 / Eq. 2 and the t_dec fit of paper_2606_12950_gb300.calibrate
against oracle/cost_model.py, which is pinned to closed forms: Llama-3-8B's
KV footprint (32 layers, 8 KV heads of 128, bf16: 128 KiB per token) and the
co-location shapes' per-layer footprints."""
import numpy as np
import pytest

import oracle.cost_model as CM
from paper_2606_12950_gb300 import calibrate as C


def test_oracle_alpha_closed_forms():
    assert CM.alpha(32, 8, 128) == 128 * 1024          # Llama-3-8B, bf16
    assert CM.alpha(1, 32, 128) == 16384                 # MHA 32 x 128 layer
    assert CM.alpha(1, 8, 128) == 4096                   # GQA 8 x 128 layer
    assert CM.alpha(1, 8, 128, elem_bytes=1) == 2048     # fp8 cache halves it
    assert CM.alpha(0, 8, 128) == 0


def test_oracle_equations_closed_forms():
    # a 1000-token prompt and 300 predicted tokens on Llama-3-8B: 1300 x 128 KiB
    assert CM.kv_demand(CM.alpha(32, 8, 128), 1000, 300) == 1300 * 131072
    assert CM.exec_time(0.25, 0.02, 300) == pytest.approx(6.25)
    assert CM.exec_time(0.25, 0.02, 0) == 0.25  # no output: prefill only


@pytest.mark.parametrize("layers,Hkv,d,eb", [(32, 8, 128, 2), (1, 32, 128, 2), (40, 8, 128, 2), (28, 4, 64, 1)])
def test_library_matches_oracle(layers, Hkv, d, eb):
    a = C.alpha_bytes(Hkv, d, layers, eb)
    assert a == CM.alpha(layers, Hkv, d, eb)
    for P, L in [(0, 0), (512, 17.5), (20000, 4096)]:
        assert C.kv_demand(a, P, L) == CM.kv_demand(a, P, L)
        assert C.exec_time(0.1, 0.015, L) == CM.exec_time(0.1, 0.015, L)


def test_fit_recovers_known_costs():
    """Timings generated from known costs (plus 1% noise) over the
    calibration grid: the fit returns them and t_dec scales with layers."""
    rng = np.random.default_rng(0)
    true = {"c0": 6e-6, "c_seq": 4e-8, "c_byte": 1 / 6.0e12}
    a = C.alpha_bytes(8, 128)
    samples = []
    for B in C.BATCHES:
        for n in C.CONTEXTS:
            t = C.t_layer(true, B, n, a) * (1 + 0.01 * rng.standard_normal())
            samples.append((B, n, a, t))
    coef, r2 = C.fit(samples)
    assert r2 > 0.999
    assert coef["c_byte"] == pytest.approx(true["c_byte"], rel=0.03)
    assert coef["c0"] == pytest.approx(true["c0"], rel=0.3, abs=1e-6)
    assert C.t_dec(coef, 32, 2048, a, 32) == pytest.approx(32 * C.t_layer(coef, 32, 2048, a))
    # Eq. 1 with the fitted per-token latency
    td = C.t_dec(coef, 32, 2048, a, 32)
    assert C.exec_time(0.2, td, 300) == pytest.approx(CM.exec_time(0.2, td, 300))
