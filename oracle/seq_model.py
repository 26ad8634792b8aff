"""Reference model of a sequence table's slot bookkeeping (TEST
INFRASTRUCTURE ONLY).

Per slot it tracks the number of blocks held and the length, following the
per-stage provisioning the paper describes: a stage of P + L^ tokens reserves
ceil((P + L^) / bs) blocks (Eq. 2); when the true output outruns the
prediction the reservation grows one block at a time; a shared prefix is held
by reference; blocks return to the pool at the end of a stage (trim) or of a
sequence (release) (§III-C).  Which block ids are used is the library's
business; the model fixes the counts.
"""
from __future__ import annotations


class SeqModel:
    def __init__(self, S: int, max_blocks: int, bs: int):
        self.S, self.max_blocks, self.bs = S, max_blocks, bs
        self.held = [0] * S
        self.len = [0] * S
        self.misses = 0

    def reserve(self, s: int, tokens: int) -> int:
        """Blocks the call must allocate (0 if the reservation already covers it)."""
        need = -(-tokens // self.bs)
        if need > self.max_blocks:
            raise ValueError("beyond max_blocks")
        extra = max(0, need - self.held[s])
        self.held[s] = max(self.held[s], need)
        return extra

    def share_prefix(self, dst: int, src: int, nb: int) -> None:
        if self.held[dst] or self.len[dst] or self.held[src] < nb:
            raise ValueError("bad share")
        self.held[dst] = nb

    def set_len(self, s: int, n: int) -> None:
        if not 0 <= n <= self.held[s] * self.bs:
            raise ValueError("bad length")
        self.len[s] = n

    def advance(self, seqs=None) -> list[int]:
        """Slots that grow by one block; lengths all += 1."""
        seqs = [s for s in range(self.S) if self.len[s] > 0] if seqs is None else list(seqs)
        grow = [s for s in seqs if self.len[s] + 1 > self.held[s] * self.bs]
        for s in grow:
            if self.held[s] + 1 > self.max_blocks:
                raise ValueError("beyond max_blocks")
        for s in grow:
            self.held[s] += 1
        for s in seqs:
            self.len[s] += 1
        self.misses += len(grow)
        return grow

    def release(self, s: int) -> int:
        h = self.held[s]
        self.held[s] = 0
        self.len[s] = 0
        return h

    def trim(self, s: int) -> int:
        keep = -(-self.len[s] // self.bs)
        freed = max(0, self.held[s] - keep)
        self.held[s] = min(self.held[s], keep) if self.held[s] > keep else self.held[s]
        return freed
