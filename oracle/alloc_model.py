"""Reference model of the KV pool's block accounting (TEST INFRASTRUCTURE ONLY).

The paper's node runtime hands KV pages of one shared pool out per stage,
reserving alpha(M) * (P + L^) of KV per stage (Eq. 2, i.e. ceil((P + L^)/bs)
blocks), keeps explicit accounting M_kv + M_res <= M_total, and rejects a
stage whose memory cannot be provided instead of failing (§III-C).  Which
physical ids a request receives is the library's policy, not the paper's; what
this model fixes is what must hold for any correct allocator with the stated
slab policy:

  * pages are grouped in superpages of K = max_L k_L pages; a layout whose
    free list is empty takes one whole free superpage and cuts it into K/k_L
    blocks; freed blocks stay with their layout;
  * so a request for n blocks of layout L succeeds iff
        n <= cached_L + unassigned_superpages * (K / k_L),
    and on failure nothing changes;
  * a returned block id is k_L-aligned inside a superpage, not live before the
    call, and starts with refcount 1; ids of one call are distinct;
  * a reference drop frees the block when its count reaches zero; dropping
    more references than a block holds, or naming a block of another layout,
    is rejected with no change.

The model keeps counts and refcounts only and checks ids for validity; it
never predicts which ids come back.
"""
from __future__ import annotations

from collections import Counter


class AllocModel:
    def __init__(self, n_pages: int, pages_per_block: list[int]):
        self.K = max(pages_per_block)
        self.k = list(pages_per_block)
        self.n_super = n_pages // self.K
        self.unassigned = self.n_super
        self.cached = [0] * len(self.k)
        self.ref: dict[int, int] = {}
        self.owner: dict[int, int] = {}

    def capacity(self, layout: int) -> int:
        return self.cached[layout] + self.unassigned * (self.K // self.k[layout])

    def alloc(self, layout: int, n: int, ids) -> bool:
        """Apply an allocation that the library answered with ``ids`` (None =
        refused).  Returns whether the model agrees with the answer."""
        can = n <= self.capacity(layout)
        if ids is None:
            return not can
        if not can or len(ids) != n or len(set(ids)) != n:
            return False
        for i in ids:
            if i in self.ref or i % self.k[layout] != 0 or not (0 <= i < self.n_super * self.K):
                return False
        need = n
        take = min(need, self.cached[layout])
        self.cached[layout] -= take
        need -= take
        per = self.K // self.k[layout]
        while need > 0:
            self.unassigned -= 1
            self.cached[layout] += per
            t = min(need, self.cached[layout])
            self.cached[layout] -= t
            need -= t
        for i in ids:
            self.ref[i] = 1
            self.owner[i] = layout
        return True

    def free_ok(self, layout: int, ids) -> bool:
        c = Counter(ids)
        return all(i in self.ref and self.owner[i] == layout and c[i] <= self.ref[i] for i in c)

    def free(self, layout: int, ids) -> None:
        for i in ids:
            self.ref[i] -= 1
            if self.ref[i] == 0:
                del self.ref[i]
                del self.owner[i]
                self.cached[layout] += 1

    def ref_ok(self, layout: int, ids) -> bool:
        return all(i in self.ref and self.owner[i] == layout for i in ids)

    def add_ref(self, ids) -> None:
        for i in ids:
            self.ref[i] += 1

    def used(self, layout: int) -> int:
        return sum(1 for i, o in self.owner.items() if o == layout)
