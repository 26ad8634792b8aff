"""Reference statement of the paper's cost translation (TEST INFRASTRUCTURE
ONLY: tests use it; the library never does).

  * Eq. 1: the execution-time estimate of a stage is its prefill latency for
    prompt length P plus the average per-token decode latency times the
    predicted output length:  T_exec = t_pre(P, M) + t_dec(M) * L_hat.
  * Eq. 2: its KV demand is the model's per-token KV footprint times the
    tokens it will hold:  R_kv = alpha(M) * (P + L_hat).
  * alpha(M) for a decoder whose layers each cache one K and one V vector
    per KV head: layers * 2 * Hkv * d * bytes per element.
"""


def alpha(layers: int, n_kv_heads: int, head_dim: int, elem_bytes: int = 2) -> int:
    total = 0
    for _ in range(layers):
        total += 2 * n_kv_heads * head_dim * elem_bytes  # K and V of every KV head
    return total


def exec_time(t_pre: float, t_dec: float, L_hat: float) -> float:
    """Eq. 1."""
    return t_pre + t_dec * L_hat


def kv_demand(alpha_bytes: int, P: int, L_hat: float) -> float:
    """Eq. 2."""
    return alpha_bytes * (P + L_hat)
