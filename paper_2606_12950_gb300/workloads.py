"""Seeded synthetic inputs for paged decode attention.

This module only draws numbers: context lengths, physical block placements,
bf16 query/key/value values and step schedules.  It holds none of the
attention or append arithmetic, so both the CUDA path and the fp64 oracle can
take their inputs from it without sharing any of the method.

The paper's workload trace (nine multi-agent applications, §IV-A, Table 1) is
not available, so these generators stand in for it with the shapes the paper
describes: heavy-tailed output lengths (§II, Observation 1), agent chains whose
context grows stage by stage (§I, §III-B), and several co-located models
sharing one KV pool (§III-C, Table 5).

All floating-point values are fp32 N(0, 1) draws rounded to bf16 with
round-to-nearest-even, returned as raw uint16 bit patterns.
"""
from __future__ import annotations

import math
from dataclasses import dataclass, field

import numpy as np

BF16 = np.uint16


# ---------------------------------------------------------------------------
# value generation
# ---------------------------------------------------------------------------
def bf16_bits_from_f32(x: np.ndarray) -> np.ndarray:
    """Round fp32 values to bf16 (round to nearest, ties to even); return the bits.

    Inputs here are finite normal draws, so NaN/Inf handling is not needed.
    """
    u = np.ascontiguousarray(x, dtype=np.float32).view(np.uint32)
    rounded = (u + np.uint32(0x7FFF) + ((u >> np.uint32(16)) & np.uint32(1))) >> np.uint32(16)
    return rounded.astype(BF16)


def bf16_bits_to_f64(b: np.ndarray) -> np.ndarray:
    """Widen bf16 bit patterns exactly to fp64."""
    u = np.asarray(b, dtype=np.uint16).astype(np.uint32) << np.uint32(16)
    return u.view(np.float32).astype(np.float64)


def bf16_normal(rng: np.random.Generator, shape) -> np.ndarray:
    """bf16 bits of fp32 N(0,1) draws."""
    return bf16_bits_from_f32(rng.standard_normal(size=shape, dtype=np.float32))


def bf16_normal_fill(out: np.ndarray, seed: int, chunk_elems: int = 1 << 24) -> None:
    """Fill a large uint16 array with bf16 N(0,1) bits in independent seeded chunks.

    Chunk i draws from ``np.random.default_rng([seed, i])`` so the content of a
    chunk does not depend on how many chunks precede it; the chunks are filled
    by a thread pool (numpy releases the GIL while drawing).
    """
    flat = out.reshape(-1)
    n = flat.size
    nchunks = (n + chunk_elems - 1) // chunk_elems

    def work(i: int) -> None:
        lo = i * chunk_elems
        hi = min(n, lo + chunk_elems)
        r = np.random.default_rng([seed, i])
        flat[lo:hi] = bf16_bits_from_f32(r.standard_normal(size=hi - lo, dtype=np.float32))

    if nchunks <= 1:
        for i in range(nchunks):
            work(i)
        return
    from concurrent.futures import ThreadPoolExecutor
    import os

    workers = max(1, min(16, len(os.sched_getaffinity(0))))
    with ThreadPoolExecutor(max_workers=workers) as ex:
        list(ex.map(work, range(nchunks)))


# ---------------------------------------------------------------------------
# length distributions
# ---------------------------------------------------------------------------
def lognormal_lengths(rng, n: int, median: float, sigma: float, lo: int, hi: int) -> np.ndarray:
    """round(median * exp(sigma * N(0,1))), clipped to [lo, hi]."""
    z = rng.standard_normal(size=n)
    x = np.rint(median * np.exp(sigma * z))
    return np.clip(x, lo, hi).astype(np.int64)


def bounded_pareto_lengths(rng, n: int, alpha: float, lo: int, hi: int) -> np.ndarray:
    """Truncated Pareto(alpha) on [lo, hi] by inverse CDF, floored to integers."""
    u = rng.random(size=n)
    x = lo / np.power(1.0 - u * (1.0 - (lo / hi) ** alpha), 1.0 / alpha)
    return np.clip(np.floor(x), lo, hi).astype(np.int64)


# ---------------------------------------------------------------------------
# one batch in one layout
# ---------------------------------------------------------------------------
@dataclass
class Batch:
    """A decode batch of one layout inside a block-paged pool.

    ``pool`` is the whole pool as uint16 (bf16 bits), ``page_elems`` bf16
    elements per page; a block of this layout starts at ``table[s][i] *
    page_elems`` and is laid out as ``[K|V][Hkv][bs][d]``.
    ``ctx_lens`` are post-append lengths (the token appended this step is the
    last one).
    """

    S: int
    Hq: int
    Hkv: int
    d: int
    bs: int
    max_blocks: int
    page_elems: int
    n_pages: int
    ctx_lens: np.ndarray  # int32 [S], post-append
    table: np.ndarray  # int32 [S, max_blocks]
    q: np.ndarray  # uint16 [S, Hq, d]
    k_new: np.ndarray  # uint16 [S, Hkv, d]
    v_new: np.ndarray  # uint16 [S, Hkv, d]
    pool: np.ndarray | None = None  # uint16 [n_pages * page_elems]
    scale: float = 0.0
    meta: dict = field(default_factory=dict)

    @property
    def G(self) -> int:
        return self.Hq // self.Hkv

    @property
    def block_elems(self) -> int:
        return 2 * self.Hkv * self.bs * self.d


def share_prefix(b: "Batch", groups) -> "Batch":
    """Make each group's members hold their first ``tokens`` tokens in the same
    physical blocks as the group's first member (a prefix shared by
    reference); ``groups`` = [(members, tokens), ...], tokens a multiple of
    the block size.  The members' own blocks for those positions become
    unused.  Returns ``b`` with its table changed in place."""
    for members, tokens in groups:
        assert tokens % b.bs == 0
        nb = tokens // b.bs
        lead = int(members[0])
        for s in members[1:]:
            b.table[int(s), :nb] = b.table[lead, :nb]
    return b


def make_batch(
    seed: int,
    pre_lens,
    Hq: int,
    Hkv: int,
    d: int,
    bs: int,
    n_pages: int | None = None,
    page_elems: int | None = None,
    extra_blocks: int = 0,
    table_tokens=None,
    max_blocks: int | None = None,
    fill_pool: bool = True,
    pool_fill: str = "normal",
) -> Batch:
    """Draw a batch: placements, pool contents, q, and the K/V rows to append.

    ``pre_lens`` are the cached lengths before this step; the batch's
    ``ctx_lens`` add the one appended token.  Each sequence's table covers
    ``table_tokens[s]`` tokens (default: its post-append length).  Physical
    blocks are a seeded random sample (without replacement) of the pool's
    block slots, so the placement is scrambled.  Table entries past a
    sequence's last block are -1 (never read).
    """
    rng = np.random.default_rng(seed)
    pre = np.asarray(pre_lens, dtype=np.int64)
    S = int(pre.size)
    ctx = pre + 1
    cover = ctx if table_tokens is None else np.maximum(np.asarray(table_tokens, np.int64), ctx)
    nblk = (cover + bs - 1) // bs
    if max_blocks is None:
        max_blocks = int(max(1, nblk.max(initial=1)))
    block_elems = 2 * Hkv * bs * d
    if page_elems is None:
        page_elems = block_elems
    assert block_elems % page_elems == 0
    k = block_elems // page_elems
    need = int(nblk.sum())
    if n_pages is None:
        n_pages = (need + extra_blocks) * k
    slots = n_pages // k
    assert slots >= need, "pool too small for the batch"
    chosen = rng.permutation(slots)[:need].astype(np.int64) * k
    table = np.full((S, max_blocks), -1, dtype=np.int32)
    pos = 0
    for s in range(S):
        nb = int(nblk[s])
        table[s, :nb] = chosen[pos : pos + nb]
        pos += nb
    q = bf16_normal(rng, (S, Hq, d))
    k_new = bf16_normal(rng, (S, Hkv, d))
    v_new = bf16_normal(rng, (S, Hkv, d))
    pool = None
    if fill_pool:
        pool = np.empty(n_pages * page_elems, dtype=BF16)
        if pool_fill == "normal":
            bf16_normal_fill(pool, seed + 7919)
        elif pool_fill == "sentinel":
            pool.fill(0xFFFF)
        else:
            raise ValueError(pool_fill)
    return Batch(
        S=S, Hq=Hq, Hkv=Hkv, d=d, bs=bs, max_blocks=max_blocks,
        page_elems=page_elems, n_pages=n_pages,
        ctx_lens=ctx.astype(np.int32), table=table, q=q, k_new=k_new, v_new=v_new,
        pool=pool, scale=1.0 / math.sqrt(d),
        meta={"seed": seed, "pre_lens": pre.copy()},
    )


# ---------------------------------------------------------------------------
# the five named workloads (single-step batches; step schedules below)
# ---------------------------------------------------------------------------
def config1_tiny(seed: int = 1001) -> Batch:
    """4 sequences cached at 17/64/100/255 tokens, 4 q / 2 KV heads, d=64,
    bs=16, physical blocks permuted inside a 128-block pool."""
    return make_batch(seed, [17, 64, 100, 255], Hq=4, Hkv=2, d=64, bs=16, n_pages=128)


def config2_lengths(seed: int = 1002, S: int = 64, median: float = 1024.0,
                    sigma: float = 1.0, clip: int = 16384) -> np.ndarray:
    """Llama-3-8B-shaped layer: lognormal cached lengths (median 1024)."""
    rng = np.random.default_rng(seed)
    return lognormal_lengths(rng, S, median, sigma, 1, clip)


def config2_llama8b(seed: int = 1002, steps: int = 100, fill_pool: bool = True,
                    sigma: float = 1.0) -> Batch:
    """Llama-3-8B-shaped attention layer (32 q / 8 KV heads, d=128, bs=16),
    64 sequences; each table already holds the blocks for ``steps`` further
    appends, so the table stays fixed over the run."""
    pre = config2_lengths(seed, sigma=sigma)
    b = make_batch(seed, pre, Hq=32, Hkv=8, d=128, bs=16, extra_blocks=64,
                   table_tokens=pre + steps, fill_pool=fill_pool)
    b.meta["steps"] = steps
    b.meta["sigma"] = sigma
    return b


def step_rows(seed: int, step: int, S: int, Hq: int, Hkv: int, d: int):
    """Fresh q / k_new / v_new for decode step ``step`` (seeded per step)."""
    rng = np.random.default_rng([seed, 1, step])
    return (bf16_normal(rng, (S, Hq, d)), bf16_normal(rng, (S, Hkv, d)),
            bf16_normal(rng, (S, Hkv, d)))


# ---------------------------------------------------------------------------
# config 3: Planner -> Coder -> Reviewer agent chains
# ---------------------------------------------------------------------------
PREFIX_TOKENS = 2048  # system prompt shared by reference by every chain
CHAIN_STAGES = 3


@dataclass
class ChainDraws:
    """Random draws of one agent chain: the user prompt length, and per stage
    the true output length and the factor U[0.8, 1.5] that turns it into the
    predicted length the stage reserves for."""

    prompt: int
    out_len: np.ndarray  # int64 [CHAIN_STAGES]
    u: np.ndarray        # float64 [CHAIN_STAGES]


def chain_draws(rng: np.random.Generator, median: float = 300.0, sigma: float = 1.0,
                max_out: int = 4096) -> ChainDraws:
    prompt = int(lognormal_lengths(rng, 1, median, sigma, 1, max_out)[0])
    out_len = lognormal_lengths(rng, CHAIN_STAGES, median, sigma, 1, max_out)
    u = rng.uniform(0.8, 1.5, size=CHAIN_STAGES)
    return ChainDraws(prompt, out_len, u)


# ---------------------------------------------------------------------------
# config 4: three co-located models in one pool filled to 90%
# ---------------------------------------------------------------------------
COLOC_LAYOUTS = [(32, 32), (32, 8), (40, 8)]  # (Hq, Hkv), d = 128, bs = 16
COLOC_SPLIT = (205, 205, 102)


def config4_colocation(seed: int = 1004, fill_pool: bool = True, fill: float = 0.9):
    """Three layer shapes (MHA 32/32, GQA 32/8, GQA 40/8; d = 128, bs = 16)
    sharing one pool of 64 KiB pages; an MHA block spans 4 pages.  512
    sequences split 205/205/102 with bounded-Pareto(1.5) cached lengths on
    [128, 32768].  The pool holds the blocks the batch needs (after this
    step's append) plus free room so that it is `fill` full; blocks sit at
    seeded random places.  Returns (list of Batch sharing `pool`, n_pages,
    page_elems)."""
    rng = np.random.default_rng(seed)
    d, bs = 128, 16
    page_elems = 2 * 8 * bs * d  # 64 KiB of bf16
    lens = [bounded_pareto_lengths(rng, n, 1.5, 128, 32768) for n in COLOC_SPLIT]
    kpages = [2 * hkv * bs * d // page_elems for _, hkv in COLOC_LAYOUTS]  # 4, 1, 1
    nblk = [(l + 1 + bs - 1) // bs for l in lens]  # post-append
    need_pages = sum(int(nb.sum()) * k for nb, k in zip(nblk, kpages))
    n_super = -(-int(np.ceil(need_pages / fill)) // 4)
    n_pages = n_super * 4
    supers = rng.permutation(n_super)
    # MHA blocks take whole superpages; GQA blocks take single pages of the rest
    mha_need = int(nblk[0].sum())
    mha_ids = supers[:mha_need] * 4
    rest = np.concatenate([sp * 4 + np.arange(4) for sp in supers[mha_need:]])
    rest = rest[rng.permutation(rest.size)]
    gqa_ids = [rest[: int(nblk[1].sum())], rest[int(nblk[1].sum()) : int(nblk[1].sum()) + int(nblk[2].sum())]]
    ids = [mha_ids] + gqa_ids
    batches = []
    for li, ((Hq, Hkv), pre, nb, blk) in enumerate(zip(COLOC_LAYOUTS, lens, nblk, ids)):
        S = pre.size
        max_blocks = int(nb.max())
        table = np.full((S, max_blocks), -1, dtype=np.int32)
        pos = 0
        for s in range(S):
            table[s, : nb[s]] = blk[pos : pos + nb[s]]
            pos += int(nb[s])
        q = bf16_normal(rng, (S, Hq, d))
        k_new = bf16_normal(rng, (S, Hkv, d))
        v_new = bf16_normal(rng, (S, Hkv, d))
        batches.append(Batch(S=S, Hq=Hq, Hkv=Hkv, d=d, bs=bs, max_blocks=max_blocks, page_elems=page_elems,
                             n_pages=n_pages, ctx_lens=(pre + 1).astype(np.int32), table=table, q=q,
                             k_new=k_new, v_new=v_new, scale=1.0 / math.sqrt(d),
                             meta={"seed": seed, "layout": li, "pre_lens": pre.copy()}))
    pool = None
    if fill_pool:
        pool = np.empty(n_pages * page_elems, dtype=BF16)
        bf16_normal_fill(pool, seed + 7919)
    for b in batches:
        b.pool = pool
    return batches, n_pages, page_elems


# ---------------------------------------------------------------------------
# config 5: long-context heavy-tail stress
# ---------------------------------------------------------------------------
def config5_lengths(rng, n: int) -> np.ndarray:
    """bounded Pareto(1.2) cached lengths on [256, 131072]"""
    return bounded_pareto_lengths(rng, n, 1.2, 256, 131072)


def config5_budgets(rng, n: int, lo: int = 1, hi: int = 64) -> np.ndarray:
    """decode steps each sequence has left before it finishes (uniform)"""
    return rng.integers(lo, hi + 1, size=n)
