"""Host step schedules of the multi-step workloads, driven through the
library's sequence tables (kv_seqtab_*).

AgentChains (config 3): concurrent Planner -> Coder -> Reviewer chains.  A
2048-token system prompt is held once and shared by reference by every
chain.  Each stage reserves ceil((context + L^) / bs) blocks for its
predicted output L^ = L * U (Eq. 2); a true output L longer than L^ grows
the reservation one block per 16 tokens; at the end of a stage the KV is
kept for the next stage (stages build on the previous context) and the
unused reservation is trimmed; a finished chain is released and a new one
is admitted in its slot (§III-B, §III-C).

LongContextStress (config 5): 1024 sequences with heavy-tailed contexts;
each decodes for a drawn number of steps, then is released and replaced by
a new sequence, so freed blocks are reused in scrambled order.

Only bookkeeping happens here; the block tables and lengths go to the device
with SeqTab.sync and the kernels run through kvpool.
"""
from __future__ import annotations

import math

import numpy as np

from . import kvpool as K
from . import workloads as W


class AgentChains:
    """n_chains decode slots (rows 0 .. n_chains-1) plus one slot holding the
    shared system prompt (row n_chains, never decoded)."""

    def __init__(self, pool, layout: int, n_chains: int, max_blocks: int, bs: int, seed: int,
                 median: float = 300.0, max_out: int = 4096, prefix_tokens: int = W.PREFIX_TOKENS):
        if prefix_tokens % bs:
            raise ValueError("the shared prefix must fill whole blocks")
        self.n = n_chains
        self.bs = bs
        self.rng = np.random.default_rng(seed)
        self.median = median
        self.max_out = max_out
        self.prefix_tokens = prefix_tokens
        self.tab = K.SeqTab(pool, layout, n_chains + 1, max_blocks)
        self.prefix_slot = n_chains
        self.tab.reserve(self.prefix_slot, prefix_tokens)
        self.tab.set_len(self.prefix_slot, prefix_tokens)
        self.draws = [None] * n_chains
        self.stage = np.zeros(n_chains, dtype=np.int64)
        self.left = np.zeros(n_chains, dtype=np.int64)   # decode steps left in the current stage
        self.ctx = np.zeros(n_chains, dtype=np.int64)    # cached length (host mirror)
        self.chains_done = 0
        self.stage_ends = 0
        self.rejected = 0
        for c in range(n_chains):
            self._admit(c)

    def _reserve_stage(self, c: int) -> None:
        d = self.draws[c]
        k = int(self.stage[c])
        predicted = int(math.ceil(d.out_len[k] * d.u[k]))
        self.tab.reserve(c, int(self.ctx[c]) + predicted)
        self.left[c] = int(d.out_len[k])

    def _admit(self, c: int) -> None:
        d = W.chain_draws(self.rng, self.median, 1.0, self.max_out)
        self.draws[c] = d
        self.tab.share_prefix(c, self.prefix_slot, self.prefix_tokens // self.bs)
        self.stage[c] = 0
        self.ctx[c] = self.prefix_tokens + d.prompt  # prompt K/V: synthetic, whatever the blocks hold
        self._reserve_stage(c)
        self.tab.set_len(c, int(self.ctx[c]))

    def step(self) -> None:
        """One decode step: finish stages that ended, then every chain gains
        this step's token (lengths are post-append afterwards)."""
        for c in np.nonzero(self.left == 0)[0]:
            c = int(c)
            self.tab.trim(c)  # stage over: drop the unused reservation, keep the KV
            self.stage_ends += 1
            self.stage[c] += 1
            if self.stage[c] == W.CHAIN_STAGES:
                self.tab.release(c)
                self.chains_done += 1
                self._admit(c)
            else:
                self._reserve_stage(c)
        self.tab.advance(np.arange(self.n, dtype=np.int32))
        self.ctx += 1
        self.left -= 1

    def prefix_plan(self) -> "K.PrefixPlan":
        """Every chain holds the system prompt's blocks at the start of its
        table: one shared-prefix group over all decode rows."""
        if getattr(self, "_plan", None) is None:
            self._plan = K.PrefixPlan([(range(self.n), self.prefix_tokens)])
        return self._plan

    def close(self) -> None:
        self.tab.close()


class LongContextStress:
    """S slots with bounded-Pareto(1.2) contexts on [256, 131072]; each decodes
    for a drawn number of steps (1..64), then is released and replaced."""

    def __init__(self, pool, layout: int, S: int, max_blocks: int, seed: int):
        self.S = S
        self.rng = np.random.default_rng(seed)
        self.tab = K.SeqTab(pool, layout, S, max_blocks)
        self.left = np.zeros(S, dtype=np.int64)
        self.admitted = 0
        self.released = 0
        self.deferred = 0
        self._admit(np.arange(S))

    def _admit(self, slots: np.ndarray) -> None:
        """Release the listed slots and admit a new sequence into each, in
        one library call: a cached length and a decode budget drawn per slot,
        and a reservation for the whole run (Eq. 2 with the true length).
        Where the pool is full the admission waits (the slot stays empty and
        is retried on the next step)."""
        k = int(slots.size)
        n = W.config5_lengths(self.rng, k)
        budget = W.config5_budgets(self.rng, k)
        status = self.tab.replace(slots, n + budget, n)
        ok = status == 0
        self.left[slots[ok]] = budget[ok]
        self.admitted += int(ok.sum())
        self.deferred += k - int(ok.sum())

    def step(self) -> None:
        lens = self.tab.lens()
        done = np.nonzero(self.left == 0)[0]
        if done.size:
            self.released += int((lens[done] > 0).sum())
            self._admit(done)
            lens = self.tab.lens()
        live = np.nonzero(lens > 0)[0].astype(np.int32)
        self.tab.advance(live)
        self.left[live] -= 1

    def close(self) -> None:
        self.tab.close()
