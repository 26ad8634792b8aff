// pool_internal.h -- host-side state of a kv_pool, shared by the allocator
// (pool.cpp) and the launch wrappers (kernels.cu).  Not part of the ABI.
#pragma once

#include <atomic>
#include <cstdint>
#include <mutex>
#include <vector>

#include <cuda.h>

#include "kvpool.h"

// Physical backing of a VMM pool: the virtual range is cut into chunks that
// are mapped when the allocator needs their superpages and unmapped by
// kv_pool_trim once all their superpages are free again.
struct kv_vmm_state {
    bool active = false;        // VMM-backed pool
    bool owns_va = false;       // the library reserved the virtual range (CUDA VMM backend)
    uint64_t chunk_bytes = 0;
    int32_t supers_per_chunk = 0;
    int64_t n_chunks = 0;
    std::vector<uint8_t> mapped;           // per chunk
    std::vector<uint64_t> handle;          // per chunk: CUmemGenericAllocationHandle (CUDA backend)
    std::vector<int32_t> free_supers;      // per chunk: superpages in super_free
    std::vector<int32_t> unmapped_order;   // stack of unmapped chunks, next to map at the back
    uint64_t mapped_bytes = 0;
    uint64_t physical_limit = 0;           // 0 = none
    kv_budget *budget = nullptr;
    int (*map_fn)(void *, uint64_t, uint64_t) = nullptr;
    int (*unmap_fn)(void *, uint64_t, uint64_t) = nullptr;
    void *ctx = nullptr;
    uint64_t va_bytes = 0;                 // reserved size (CUDA backend)
};

struct kv_pool {
    kv_pool_desc desc;
    uint64_t page_bytes = 0;
    int64_t n_pages = 0;
    int32_t super_pages = 1;                  // K: pages per superpage
    int32_t pages_per_block[KV_MAX_LAYOUTS];  // k_L
    uint64_t block_bytes[KV_MAX_LAYOUTS];
    std::vector<int32_t> super_free;          // stack of free superpage indices
    std::vector<int32_t> free_blocks[KV_MAX_LAYOUTS];  // LIFO stacks of block ids
    std::vector<int32_t> refcnt;              // per page id (block start); 0 = not live
    std::vector<int8_t> owner;                // layout owning the block at page id, -1 none
    std::vector<int32_t> tally;               // per page id, all 0 between calls: duplicate counts of a free
    int64_t used_blocks[KV_MAX_LAYOUTS];
    int64_t carved_blocks[KV_MAX_LAYOUTS];    // blocks cut from superpages so far
    int device = 0;
    int sm_count = 0;
    int attn_variant = 0;
    bool step_overlap = false;                // kv_set_attn_step_overlap
    std::atomic<int64_t> overlapped{0};       // calls that overlapped the previous combine
    CUtensorMap tmap[KV_MAX_LAYOUTS];        // pool viewed as rows of d bf16, per layout
    bool tmap_ok[KV_MAX_LAYOUTS] = {false, false, false, false};
    kv_vmm_state vmm;
    uint64_t shuffle_state = 0;               // splitmix64 state for placing newly mapped superpages
    std::vector<kv_seqtab *> seqtabs;         // live sequence tables over this pool (detached on destroy)
    std::mutex mu;
};

// VMM backend (vmm.cpp); called with the pool's mutex held.
int kvp_vmm_map_chunk(kv_pool *p);                  // map the next unmapped chunk
int kvp_vmm_unmap_chunk(kv_pool *p, int64_t chunk);  // unmap a chunk whose superpages are all free
void kvp_vmm_release_all(kv_pool *p);                // on destroy

// Called by kv_pool_destroy, with the pool's mutex held, for every sequence
// table still open over the pool (seqtab.cpp).
void kvp_seqtab_detach(kv_seqtab *t);

// Resolve the allocation-free attention's scratch on `device`, the current
// device (noalloc.cu); called when a pool is created on a visible GPU.
void kvp_noalloc_prepare(int device);

// Validate that a block id is a whole block of layout L inside the pool.
// In a VMM pool the block must also lie in a mapped chunk.
inline bool kvp_block_in_pool(const kv_pool *p, int layout, int64_t id)
{
    if (id < 0) return false;
    if ((uint64_t)id * p->page_bytes + p->block_bytes[layout] > (uint64_t)p->n_pages * p->page_bytes) return false;
    if (p->vmm.active) {
        const int64_t c = id / ((int64_t)p->super_pages * p->vmm.supers_per_chunk);
        if (!p->vmm.mapped[(size_t)c]) return false;
    }
    return true;
}
