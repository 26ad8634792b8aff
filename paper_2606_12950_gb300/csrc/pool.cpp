// pool.cpp -- host-side manager of the shared block-paged KV pool.
//
// The paper's node runtime keeps one shared KV pool per GPU and hands pages
// out to stages on demand, rejecting a stage whose memory cannot be mapped
// rather than failing (§III-C, "Spatial multiplexing with virtual-memory KV
// cache"); per stage it reserves alpha(M) * (P + L^) of KV (Eq. 2), i.e.
// ceil((P + L^) / bs) blocks here.  This file is that allocator for a fixed
// caller-owned device buffer: a slab scheme over superpages so layouts of
// different block sizes (co-located models, Table 5) share one pool.
#include <algorithm>
#include <cstring>
#include <unordered_map>

#include <cuda_runtime.h>

#include "pool_internal.h"
#include "stream_order.h"

namespace {

uint64_t splitmix64(uint64_t &state)
{
    uint64_t z = (state += 0x9E3779B97F4A7C15ull);
    z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
    z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
    return z ^ (z >> 31);
}

bool layout_ok(const kv_pool *p, int layout)
{
    return p && layout >= 0 && layout < p->desc.num_layouts;
}

// Take one free superpage and cut it into blocks of `layout`, pushed so that
// they pop in ascending order.
bool carve(kv_pool *p, int layout)
{
    if (p->super_free.empty()) return false;
    int32_t sp = p->super_free.back();
    p->super_free.pop_back();
    if (p->vmm.active) p->vmm.free_supers[(size_t)(sp / p->vmm.supers_per_chunk)] -= 1;
    int32_t k = p->pages_per_block[layout];
    int32_t nb = p->super_pages / k;
    int64_t first = (int64_t)sp * p->super_pages;
    for (int32_t j = nb - 1; j >= 0; --j) p->free_blocks[layout].push_back((int32_t)(first + (int64_t)j * k));
    p->carved_blocks[layout] += nb;
    return true;
}

}  // namespace

extern "C" {

const char *kv_version(void) { return "libkvpool 0.1 (sm_103a)"; }

int kv_pool_create(const kv_pool_desc *desc, kv_pool **out_pool)
{
    if (!desc || !out_pool) return KV_ERR_INVALID_ARG;
    *out_pool = nullptr;
    if (!desc->device_base || ((uintptr_t)desc->device_base & 255u)) return KV_ERR_INVALID_ARG;
    if (!desc->device_error || ((uintptr_t)desc->device_error & 3u)) return KV_ERR_INVALID_ARG;
    if (desc->num_layouts < 1 || desc->num_layouts > KV_MAX_LAYOUTS) return KV_ERR_INVALID_ARG;
    if (desc->block_size < 1 || desc->block_size > 256) return KV_ERR_INVALID_ARG;
    uint64_t min_block = UINT64_MAX, max_block = 0;
    for (int l = 0; l < desc->num_layouts; ++l) {
        const kv_layout &L = desc->layouts[l];
        if (L.num_kv_heads < 1 || L.num_kv_heads > 1024) return KV_ERR_INVALID_ARG;
        if (L.head_dim < 8 || L.head_dim > 512 || (L.head_dim % 8)) return KV_ERR_INVALID_ARG;
        uint64_t bb = 2ull * L.num_kv_heads * desc->block_size * L.head_dim * 2ull;
        min_block = std::min(min_block, bb);
        max_block = std::max(max_block, bb);
    }
    uint64_t page = desc->page_bytes ? desc->page_bytes : min_block;
    if (page == 0 || (page % 256)) return KV_ERR_INVALID_ARG;
    kv_pool *p = new kv_pool();
    p->desc = *desc;
    p->page_bytes = page;
    p->n_pages = (int64_t)(desc->pool_bytes / page);
    if (p->n_pages > INT32_MAX) { delete p; return KV_ERR_INVALID_ARG; }
    int32_t K = 1;
    for (int l = 0; l < desc->num_layouts; ++l) {
        const kv_layout &L = desc->layouts[l];
        uint64_t bb = 2ull * L.num_kv_heads * desc->block_size * L.head_dim * 2ull;
        if (bb % page) { delete p; return KV_ERR_INVALID_ARG; }
        p->block_bytes[l] = bb;
        p->pages_per_block[l] = (int32_t)(bb / page);
        K = std::max<int32_t>(K, p->pages_per_block[l]);
    }
    for (int l = 0; l < desc->num_layouts; ++l) {
        if (K % p->pages_per_block[l]) { delete p; return KV_ERR_INVALID_ARG; }
        p->used_blocks[l] = 0;
        p->carved_blocks[l] = 0;
    }
    p->super_pages = K;
    int64_t n_super = p->n_pages / K;
    if (n_super < 1) { delete p; return KV_ERR_INVALID_ARG; }
    // free stack: pop order ascending, or a seeded permutation
    std::vector<int32_t> order((size_t)n_super);
    for (int64_t i = 0; i < n_super; ++i) order[(size_t)i] = (int32_t)i;
    if (desc->shuffle_seed) {
        uint64_t st = desc->shuffle_seed;
        for (int64_t i = n_super - 1; i > 0; --i) {
            int64_t j = (int64_t)(splitmix64(st) % (uint64_t)(i + 1));
            std::swap(order[(size_t)i], order[(size_t)j]);
        }
    }
    p->super_free.assign(order.rbegin(), order.rend());
    p->refcnt.assign((size_t)p->n_pages, 0);
    p->owner.assign((size_t)p->n_pages, (int8_t)-1);
    p->tally.assign((size_t)p->n_pages, 0);
    if (cudaGetDevice(&p->device) != cudaSuccess ||
        cudaDeviceGetAttribute(&p->sm_count, cudaDevAttrMultiProcessorCount, p->device) != cudaSuccess) {
        // host-only use (no GPU visible): allocation still works; launches will fail
        cudaGetLastError();
        p->sm_count = 0;
    } else {
        // the allocation-free attention's fixed scratch is taken on this
        // device now, before the caller fills it with KV blocks
        kvp_noalloc_prepare(p->device);
    }
    *out_pool = p;
    return KV_OK;
}

int kv_pool_destroy(kv_pool *pool)
{
    if (!pool) return KV_ERR_INVALID_ARG;
    {
        // sequence tables still open lose their pool: their blocks end with it
        std::lock_guard<std::mutex> g(pool->mu);
        for (kv_seqtab *t : pool->seqtabs) kvp_seqtab_detach(t);
        pool->seqtabs.clear();
    }
    if (pool->vmm.active) kvp_vmm_release_all(pool);
    delete pool;
    return KV_OK;
}

int kv_alloc_blocks(kv_pool *p, int layout, int n, int32_t *out_ids)
{
    if (!layout_ok(p, layout) || n < 0 || (n > 0 && !out_ids)) return KV_ERR_INVALID_ARG;
    std::lock_guard<std::mutex> g(p->mu);
    int32_t k = p->pages_per_block[layout];
    // capacity check first so the call is all-or-nothing; a VMM pool maps the
    // chunks it lacks before anything is allocated (a chunk that cannot be
    // mapped rejects the request; chunks mapped so far stay as free capacity)
    const int64_t per_super = p->super_pages / k;
    int64_t avail = (int64_t)p->free_blocks[layout].size() + (int64_t)p->super_free.size() * per_super;
    if (avail < n) {
        if (!p->vmm.active) return KV_ERR_OUT_OF_BLOCKS;
        const int64_t supers = (n - avail + per_super - 1) / per_super;
        const int64_t chunks = (supers + p->vmm.supers_per_chunk - 1) / p->vmm.supers_per_chunk;
        if (chunks > (int64_t)p->vmm.unmapped_order.size()) return KV_ERR_OUT_OF_BLOCKS;
        for (int64_t c = 0; c < chunks; ++c)
            if (kvp_vmm_map_chunk(p) != KV_OK) return KV_ERR_OUT_OF_BLOCKS;
    }
    for (int i = 0; i < n; ++i) {
        if (p->free_blocks[layout].empty()) carve(p, layout);
        int32_t id = p->free_blocks[layout].back();
        p->free_blocks[layout].pop_back();
        p->refcnt[(size_t)id] = 1;
        p->owner[(size_t)id] = (int8_t)layout;
        out_ids[i] = id;
    }
    p->used_blocks[layout] += n;
    return KV_OK;
}

static int check_live(kv_pool *p, int layout, int n, const int32_t *ids, bool for_free)
{
    // a free may name an id at most refcnt times: counted in the pool's
    // per-page tally, which is back to all zeros when the check returns
    int rc = KV_OK;
    int i = 0;
    for (; i < n; ++i) {
        int32_t id = ids[i];
        if (id < 0 || id >= p->n_pages) { rc = KV_ERR_INVALID_ARG; break; }
        if (p->owner[(size_t)id] != layout || p->refcnt[(size_t)id] <= 0) { rc = KV_ERR_INVALID_ARG; break; }
        if (for_free) {
            if (++p->tally[(size_t)id] > p->refcnt[(size_t)id]) { rc = KV_ERR_INVALID_ARG; ++i; break; }
        } else if (p->refcnt[(size_t)id] == INT32_MAX) {
            rc = KV_ERR_INVALID_ARG;
            break;
        }
    }
    if (for_free)
        for (int j = 0; j < i; ++j) p->tally[(size_t)ids[j]] = 0;
    return rc;
}

int kv_free_blocks(kv_pool *p, int layout, int n, const int32_t *ids)
{
    if (!layout_ok(p, layout) || n < 0 || (n > 0 && !ids)) return KV_ERR_INVALID_ARG;
    std::lock_guard<std::mutex> g(p->mu);
    int rc = check_live(p, layout, n, ids, true);
    if (rc) return rc;
    for (int i = 0; i < n; ++i) {
        int32_t id = ids[i];
        if (--p->refcnt[(size_t)id] == 0) {
            p->owner[(size_t)id] = -1;
            p->free_blocks[layout].push_back(id);
            p->used_blocks[layout] -= 1;
        }
    }
    return KV_OK;
}

int kv_block_ref(kv_pool *p, int layout, int n, const int32_t *ids)
{
    if (!layout_ok(p, layout) || n < 0 || (n > 0 && !ids)) return KV_ERR_INVALID_ARG;
    std::lock_guard<std::mutex> g(p->mu);
    int rc = check_live(p, layout, n, ids, false);
    if (rc) return rc;
    for (int i = 0; i < n; ++i) p->refcnt[(size_t)ids[i]] += 1;
    return KV_OK;
}

int kv_block_refcount(const kv_pool *p, int32_t id, int32_t *out_count)
{
    if (!p || !out_count || id < 0 || id >= p->n_pages) return KV_ERR_INVALID_ARG;
    *out_count = p->refcnt[(size_t)id];
    return KV_OK;
}

int kv_pool_stats(const kv_pool *p, kv_stats *out)
{
    if (!p || !out) return KV_ERR_INVALID_ARG;
    std::memset(out, 0, sizeof *out);
    kv_pool *mp = const_cast<kv_pool *>(p);
    std::lock_guard<std::mutex> g(mp->mu);
    out->pages_total = p->n_pages;
    const int64_t unmapped_supers =
        p->vmm.active ? (int64_t)p->vmm.unmapped_order.size() * p->vmm.supers_per_chunk : 0;
    out->pages_unassigned = ((int64_t)p->super_free.size() + unmapped_supers) * p->super_pages;
    out->bytes_total = (uint64_t)p->n_pages * p->page_bytes;
    for (int l = 0; l < p->desc.num_layouts; ++l) {
        out->blocks_used[l] = p->used_blocks[l];
        out->blocks_cached[l] = (int64_t)p->free_blocks[l].size();
        out->blocks_capacity[l] = p->used_blocks[l] + out->blocks_cached[l] +
                                  ((int64_t)p->super_free.size() + unmapped_supers) *
                                      (p->super_pages / p->pages_per_block[l]);
        out->bytes_used += (uint64_t)p->used_blocks[l] * p->block_bytes[l];
    }
    out->bytes_mapped = p->vmm.active ? p->vmm.mapped_bytes : out->bytes_total;
    out->attn_calls_overlapped = p->overlapped.load(std::memory_order_relaxed);
    return KV_OK;
}

int kv_pool_trim(kv_pool *p, uint64_t *released_bytes)
{
    if (!p) return KV_ERR_INVALID_ARG;
    std::lock_guard<std::mutex> g(p->mu);
    // 1. superpages whose blocks are all free in their layout's list go back
    //    to the shared free list (any layout may carve them again)
    const int64_t K = p->super_pages;
    for (int l = 0; l < p->desc.num_layouts; ++l) {
        auto &fl = p->free_blocks[l];
        if (fl.empty()) continue;
        const int32_t per_super = (int32_t)(K / p->pages_per_block[l]);
        std::unordered_map<int32_t, int32_t> cnt;
        for (int32_t id : fl) cnt[(int32_t)(id / K)] += 1;
        std::vector<int32_t> whole;
        for (auto &kv : cnt)
            if (kv.second == per_super) whole.push_back(kv.first);
        if (whole.empty()) continue;
        std::sort(whole.begin(), whole.end());
        std::vector<int32_t> keep;
        keep.reserve(fl.size());
        for (int32_t id : fl)
            if (!std::binary_search(whole.begin(), whole.end(), (int32_t)(id / K))) keep.push_back(id);
        fl.swap(keep);
        p->carved_blocks[l] -= (int64_t)whole.size() * per_super;
        for (auto it = whole.rbegin(); it != whole.rend(); ++it) {
            p->super_free.push_back(*it);
            if (p->vmm.active) p->vmm.free_supers[(size_t)(*it / p->vmm.supers_per_chunk)] += 1;
        }
    }
    // 2. a VMM pool unmaps every chunk whose superpages are all free
    uint64_t released = 0;
    if (p->vmm.active) {
        const int32_t spc = p->vmm.supers_per_chunk;
        std::vector<int64_t> chunks;
        for (int64_t c = 0; c < p->vmm.n_chunks; ++c)
            if (p->vmm.mapped[(size_t)c] && p->vmm.free_supers[(size_t)c] == spc) chunks.push_back(c);
        if (!chunks.empty()) {
            // kernels still in flight may read blocks freed on the host
            if (!p->vmm.map_fn && cudaDeviceSynchronize() != cudaSuccess) return KV_ERR_CUDA;
            std::vector<int32_t> keep;
            keep.reserve(p->super_free.size());
            for (int32_t sp : p->super_free) {
                const int64_t c = sp / spc;
                if (!std::binary_search(chunks.begin(), chunks.end(), c)) keep.push_back(sp);
            }
            p->super_free.swap(keep);
            for (int64_t c : chunks) {
                const int rc = kvp_vmm_unmap_chunk(p, c);
                if (rc) return rc;
                released += p->vmm.chunk_bytes;
            }
        }
    }
    if (released_bytes) *released_bytes = released;
    return KV_OK;
}

int kv_set_attn_variant(kv_pool *p, int variant)
{
    if (!p || variant < 0 || variant > 2) return KV_ERR_INVALID_ARG;
    p->attn_variant = variant;
    return KV_OK;
}

int kv_set_attn_step_overlap(kv_pool *p, int on)
{
    if (!p || on < 0 || on > 1) return KV_ERR_INVALID_ARG;
    p->step_overlap = on != 0;
    return KV_OK;
}

int kv_block_table_upload(kv_pool *p, int layout, const int32_t *host_table, int S, int max_blocks,
                          const int32_t *host_ctx_lens, int32_t *dev_table, int32_t *dev_ctx_lens,
                          void *stream)
{
    if (!layout_ok(p, layout) || S < 0 || max_blocks < 1) return KV_ERR_INVALID_ARG;
    if (S == 0) return KV_OK;
    if (!host_table || !host_ctx_lens || !dev_table || !dev_ctx_lens) return KV_ERR_INVALID_ARG;
    const int bs = p->desc.block_size;
    for (int s = 0; s < S; ++s) {
        int32_t n = host_ctx_lens[s];
        if (n < 0 || (int64_t)n > (int64_t)max_blocks * bs) return KV_ERR_INVALID_ARG;
        int32_t nb = (n + bs - 1) / bs;
        const int32_t *row = host_table + (int64_t)s * max_blocks;
        for (int32_t i = 0; i < nb; ++i)
            if (!kvp_block_in_pool(p, layout, row[i])) return KV_ERR_INVALID_ARG;
    }
    cudaStream_t st = (cudaStream_t)stream;
    if (cudaMemcpyAsync(dev_table, host_table, sizeof(int32_t) * (size_t)S * (size_t)max_blocks,
                        cudaMemcpyHostToDevice, st) != cudaSuccess)
        return KV_ERR_CUDA;
    if (cudaMemcpyAsync(dev_ctx_lens, host_ctx_lens, sizeof(int32_t) * (size_t)S,
                        cudaMemcpyHostToDevice, st) != cudaSuccess)
        return KV_ERR_CUDA;
    kvp_note_stream(stream, false);
    return KV_OK;
}

int kv_pool_get_error(kv_pool *p, void *stream, int32_t *host_code)
{
    if (!p || !host_code) return KV_ERR_INVALID_ARG;
    cudaStream_t st = (cudaStream_t)stream;
    if (cudaMemcpyAsync(host_code, p->desc.device_error, sizeof(int32_t), cudaMemcpyDeviceToHost, st) !=
        cudaSuccess)
        return KV_ERR_CUDA;
    if (cudaMemsetAsync(p->desc.device_error, 0, sizeof(int32_t), st) != cudaSuccess) return KV_ERR_CUDA;
    kvp_note_stream(stream, false);
    return KV_OK;
}

int kv_workspace_clear(void *workspace, size_t ws_bytes, void *stream)
{
    if (!workspace && ws_bytes) return KV_ERR_INVALID_ARG;
    if (!ws_bytes) return KV_OK;
    if (cudaMemsetAsync(workspace, 0, ws_bytes, (cudaStream_t)stream) != cudaSuccess) return KV_ERR_CUDA;
    kvp_note_stream(stream, false);
    return KV_OK;
}

}  // extern "C"
