"""Calibrated decode-latency microbenchmarks (the per-model microbenchmarks
behind Eq. 1 and Eq. 2).

Eq. 1 estimates a stage's execution time as t_pre(P, M) + t_dec(M) * L_hat
and Eq. 2 its KV demand as alpha(M) * (P + L_hat).  This module measures the
part of t_dec that this library computes -- the per-layer decode step over
the paged KV cache (fused append + attention) -- on the GPU as a function of
batch size B and context length n, and fits

    t_layer(B, n) = c0 + c_seq * B + c_byte * (B * n * alpha_layer)

(a fixed launch/prologue cost, a per-sequence cost, and the KV bytes
streamed at an effective bandwidth 1 / c_byte).  alpha(M) is exact from the
layer shape.  GEMMs, prefill and everything outside the attention layer are
the serving engine's and not measured here.

    python -m paper_2606_12950_gb300.calibrate --out calib.json
"""
from __future__ import annotations

import argparse
import json

import numpy as np

# the co-located layer shapes of the co-location workload: (Hq, Hkv, d)
SHAPES = {"mha-32x32-d128": (32, 32, 128), "gqa-32x8-d128": (32, 8, 128), "gqa-40x8-d128": (40, 8, 128)}
BATCHES = (1, 8, 32, 128)
CONTEXTS = (512, 2048, 8192)


def alpha_bytes(n_kv_heads: int, head_dim: int, layers: int = 1, elem_bytes: int = 2) -> int:
    """Eq. 2's alpha(M): bytes of K and V cached per token."""
    return layers * 2 * n_kv_heads * head_dim * elem_bytes


def exec_time(t_pre: float, t_dec: float, L_hat: float) -> float:
    """Eq. 1."""
    return t_pre + t_dec * L_hat


def kv_demand(alpha: int, P: int, L_hat: float) -> float:
    """Eq. 2."""
    return alpha * (P + L_hat)


def fit(samples):
    """Least-squares fit of t = c0 + c_seq * B + c_byte * kv_bytes over
    samples [(B, n, alpha_layer, seconds)]; returns (coef dict, R^2)."""
    A = np.array([[1.0, B, B * n * a] for B, n, a, _ in samples], dtype=np.float64)
    y = np.array([t for *_, t in samples], dtype=np.float64)
    coef, *_ = np.linalg.lstsq(A, y, rcond=None)
    pred = A @ coef
    ss_res = float(((y - pred) ** 2).sum())
    ss_tot = float(((y - y.mean()) ** 2).sum()) or 1.0
    return {"c0": float(coef[0]), "c_seq": float(coef[1]), "c_byte": float(coef[2])}, 1.0 - ss_res / ss_tot


def t_layer(coef: dict, B: int, n: float, alpha_layer: int) -> float:
    return coef["c0"] + coef["c_seq"] * B + coef["c_byte"] * B * n * alpha_layer


def t_dec(coef: dict, B: int, n: float, alpha_layer: int, layers: int) -> float:
    """Attention part of the per-token decode latency of a model with
    `layers` such layers, at batch B and mean context n."""
    return layers * t_layer(coef, B, n, alpha_layer)


def measure(Hq: int, Hkv: int, d: int, B: int, n: int, bs: int = 16, iters: int = 20, warmup: int = 3,
            seed: int = 0) -> float:
    """Seconds per fused append + attention step of one layer: B sequences
    of n cached tokens (n + 1 after the append), scattered blocks; L2 is
    flushed before every timed launch (a model's layers touch different KV)."""
    import torch

    from . import kvpool as K
    from .runner import DevicePool

    dev = torch.device("cuda")
    nb = (n + 1 + bs - 1) // bs
    block = 2 * Hkv * bs * d * 2
    pool = DevicePool(B * nb + 8, block, bs, [(Hkv, d)], shuffle_seed=seed + 1)
    g = torch.Generator(device=dev)
    g.manual_seed(seed)
    pool.buf.view(torch.bfloat16).normal_(generator=g)
    ids = K.kv_alloc_blocks(pool.handle, 0, B * nb)
    table = torch.as_tensor(ids.reshape(B, nb), device=dev).contiguous()
    lens = torch.full((B,), n + 1, dtype=torch.int32, device=dev)
    q = torch.randn((B, Hq, d), generator=g, device=dev).to(torch.bfloat16)
    kn = torch.randn((B, Hkv, d), generator=g, device=dev).to(torch.bfloat16)
    vn = torch.randn((B, Hkv, d), generator=g, device=dev).to(torch.bfloat16)
    out = torch.empty_like(q)
    ws_bytes = K.kv_workspace_bytes(pool.handle, 0, B, Hq, nb)
    ws = torch.empty(max(256, ws_bytes), dtype=torch.uint8, device=dev)
    flush = torch.empty(256 << 20, dtype=torch.uint8, device=dev)  # twice the 129 MB L2
    scale = d ** -0.5

    def call():
        # the append lands in the same slot every time: n stays fixed
        K.paged_decode_attn_append(pool.handle, 0, q, kn, vn, out, table, lens, nb, B, Hq, scale, 0, ws,
                                   ws.numel())

    for _ in range(warmup):
        call()
    evs = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(iters)]
    for a, z in evs:
        flush.zero_()
        a.record()
        call()
        z.record()
    torch.cuda.synchronize()
    err = pool.error()
    pool.close()
    if err:
        raise RuntimeError(f"device error {err} during calibration")
    return float(np.median([a.elapsed_time(z) for a, z in evs])) * 1e-3


def calibrate(shapes=None, batches=BATCHES, contexts=CONTEXTS, iters: int = 20):
    """Measure every (shape, B, n) and fit each shape; returns a JSON-ready dict."""
    shapes = shapes or SHAPES
    result = {}
    for name, (Hq, Hkv, d) in shapes.items():
        a = alpha_bytes(Hkv, d)
        samples, rows = [], []
        for B in batches:
            for n in contexts:
                t = measure(Hq, Hkv, d, B, n, iters=iters)
                samples.append((B, n, a, t))
                rows.append({"B": B, "n": n, "seconds": t, "kv_bytes": B * (n + 1) * a,
                             "gbs": B * (n + 1) * a / t / 1e9})
        coef, r2 = fit(samples)
        result[name] = {"Hq": Hq, "Hkv": Hkv, "d": d, "alpha_layer_bytes": a, "coef": coef, "r2": r2,
                        "effective_gbs": (1.0 / coef["c_byte"] / 1e9) if coef["c_byte"] > 0 else None,
                        "samples": rows}
    return result


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--out", default=None)
    ap.add_argument("--iters", type=int, default=20)
    args = ap.parse_args()
    res = calibrate(iters=args.iters)
    text = json.dumps(res, indent=1)
    if args.out:
        with open(args.out, "w") as f:
            f.write(text)
    print(text)


if __name__ == "__main__":
    main()
