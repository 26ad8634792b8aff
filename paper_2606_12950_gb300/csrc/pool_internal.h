// pool_internal.h -- host-side state of a kv_pool, shared by the allocator
// (pool.cpp) and the launch wrappers (kernels.cu).  Not part of the ABI.
#pragma once

#include <cstdint>
#include <mutex>
#include <vector>

#include <cuda.h>

#include "kvpool.h"

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
    int64_t used_blocks[KV_MAX_LAYOUTS];
    int64_t carved_blocks[KV_MAX_LAYOUTS];    // blocks cut from superpages so far
    int device = 0;
    int sm_count = 0;
    int attn_variant = 0;
    CUtensorMap tmap[KV_MAX_LAYOUTS];        // pool viewed as rows of d bf16, per layout
    bool tmap_ok[KV_MAX_LAYOUTS] = {false, false, false, false};
    std::mutex mu;
};

// Validate that a block id is a whole block of layout L inside the pool.
inline bool kvp_block_in_pool(const kv_pool *p, int layout, int64_t id)
{
    if (id < 0) return false;
    return (uint64_t)id * p->page_bytes + p->block_bytes[layout] <= (uint64_t)p->n_pages * p->page_bytes;
}
