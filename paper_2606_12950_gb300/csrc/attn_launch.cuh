// attn_launch.cuh -- host-side launch of one paged-attention instantiation:
// stage count, shared memory, grid (one CTA per resident slot unless the
// caller asks for a given number of work partitions).
#pragma once

#include <algorithm>
#include <atomic>

#include "cascade_impl.cuh"
#include "stream_order.h"

namespace kvp {

// shared memory of one CTA: up to 227 KB; the block-table window (rows of the
// CTA's units resolved in the prologue) is kRowsCap entries
constexpr size_t kSmemMax = 227 * 1024;

// Resident CTAs per SM of kernel fn at this block size and dynamic shared
// memory, queried once per (block size, shared-memory size) and cached in
// the caller's slot, one slot per kernel instantiation: the runtime query
// costs microseconds of host time on every launch.
struct OccCache {
    static constexpr int kSlots = 4;  // a call may query two shapes (its workspace's, its launch's)
    // (smem * 2048 + threads) << 8 | CTAs per SM, one word so that a reader
    // sees a key only with its own value
    std::atomic<long long> slot[kSlots] = {{-1}, {-1}, {-1}, {-1}};
    std::atomic<unsigned> next{0};
};

template <class Fn>
int cached_occupancy(Fn fn, int threads, size_t smem, int *occ, OccCache &c)
{
    const long long key = (long long)smem * 2048 + threads;
    for (int i = 0; i < OccCache::kSlots; ++i) {
        const long long w = c.slot[i].load(std::memory_order_relaxed);
        if (w >= 0 && (w >> 8) == key) {
            *occ = (int)(w & 255);
            return KV_OK;
        }
    }
    int o = 0;
    if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&o, fn, threads, smem) != cudaSuccess) return KV_ERR_CUDA;
    const unsigned i = c.next.fetch_add(1, std::memory_order_relaxed) % OccCache::kSlots;
    c.slot[i].store(key << 8 | (long long)(o & 255), std::memory_order_relaxed);
    *occ = o;
    return KV_OK;
}

// what: kLaunchQuery (only *P_out), kLaunchBoth (attention, then combine),
// kLaunchAttention, kLaunchCombine
enum { kLaunchQuery = 0, kLaunchBoth = 1, kLaunchAttention = 2, kLaunchCombine = 3 };

template <int D, int G, class Comp>
int attn_run(const CUtensorMap *tmap, AttnArgs a, int P_req, int sm_count, cudaStream_t st, int what, int *P_out)
{
    auto fn = paged_attn_kernel<D, G, Comp>;
    static std::atomic<bool> attr_set{false};
    if (!attr_set.load()) {
        if (cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kSmemMax) != cudaSuccess)
            return KV_ERR_CUDA;
        attr_set.store(true);
    }
    // six warps a CTA, eight beside the shared-prefix kernel (kPlainWarps)
    a.nwarps = a.skip != nullptr ? kWarps : kPlainWarps;
    const size_t smem = attn_smem_bytes<D, G>(a.S, kRowsCap, a.nwarps);
    if (smem > kSmemMax) return KV_ERR_INVALID_ARG;  // S too large for the per-CTA sequence index
    int occ = 0;
    static OccCache occ_cache;
    if (cached_occupancy(fn, a.nwarps * 32, smem, &occ, occ_cache) != KV_OK) return KV_ERR_CUDA;
    const int P = P_req > 0 ? P_req : std::max(1, occ) * std::max(1, sm_count);
    *P_out = P;
    if (what == kLaunchQuery) return KV_OK;
    a.rows_cap = kRowsCap;
    a.P = P;
    // both kernels are programmatic dependents of what precedes them in the
    // stream: they may be scheduled early and wait on the device
    // (griddepcontrol.wait) for the previous grid to complete
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3((unsigned)P);
    cfg.blockDim = dim3((unsigned)(a.nwarps * 32));
    cfg.dynamicSmemBytes = smem;
    cfg.stream = st;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    if (what != kLaunchCombine) {
        if (cudaLaunchKernelEx(&cfg, fn, *tmap, a) != cudaSuccess) return KV_ERR_CUDA;
        kvp_note_stream(st, false);
    }
    if (what == kLaunchAttention) return KV_OK;
    CombineArgs c{a.out, a.ws_run, a.ws_part, a.S, a.Hkv, a.skip, a.ws_pre, a.KS};
    cudaLaunchConfig_t ccfg = cfg;
    // records per run: at most P * nwarps parts spread over the runs, plus
    // the prefix records in shared-prefix mode
    const double per_run = (double)P * a.nwarps / std::max(1, a.S * a.Hkv) + 1.0 + (a.skip ? a.KS : 0);
    const int groups = combine_groups<D, G>(per_run, a.skip != nullptr);
    ccfg.gridDim = dim3((unsigned)(a.S * a.Hkv));
    if constexpr (G * D / 4 >= 128) {
        // one group in shared-prefix mode: two columns a thread, so that
        // every member run fits in one wave
        if (groups == 1 && a.skip != nullptr) {
            ccfg.blockDim = dim3((unsigned)CombineShape<D, G, 2>::NCT);
            ccfg.dynamicSmemBytes = 0;
            if (cudaLaunchKernelEx(&ccfg, combine_kernel<D, G, 2>, c) != cudaSuccess) return KV_ERR_CUDA;
            kvp_note_stream(st, true);
            return KV_OK;
        }
    }
    const int threads = groups * (G * D / 4);
    ccfg.blockDim = dim3((unsigned)threads);
    ccfg.dynamicSmemBytes = combine_smem_bytes<D, G, 1>(threads);
    if (cudaLaunchKernelEx(&ccfg, combine_kernel<D, G, 1>, c) != cudaSuccess) return KV_ERR_CUDA;
    kvp_note_stream(st, true);
    return KV_OK;
}

// Shared-prefix kernel: with launch = false only reports the CTAs that fit
// on the GPU at once (occupancy x SMs) in *P_out.
template <int D, int G>
int cascade_run(const CUtensorMap *tmap, const CascadeArgs *c, int grid, int sm_count, cudaStream_t st, bool launch,
                int *P_out)
{
    auto fn = cascade_prefix_kernel<D, G>;
    const size_t smem = cascade_smem_bytes<D>();
    static std::atomic<bool> attr_set{false};
    if (!attr_set.load()) {
        if (cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem) != cudaSuccess)
            return KV_ERR_CUDA;
        attr_set.store(true);
    }
    if (!launch) {
        int occ = 0;
        static OccCache occ_cache;
        if (cached_occupancy(fn, kPreThreads, smem, &occ, occ_cache) != KV_OK) return KV_ERR_CUDA;
        *P_out = std::max(1, occ) * std::max(1, sm_count);
        return KV_OK;
    }
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3((unsigned)grid);
    cfg.blockDim = dim3(kPreThreads);
    cfg.dynamicSmemBytes = smem;
    cfg.stream = st;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    if (cudaLaunchKernelEx(&cfg, fn, *tmap, *c) != cudaSuccess) return KV_ERR_CUDA;
    kvp_note_stream(st, false);
    return KV_OK;
}

}  // namespace kvp

// one entry per head dim; variant 1 = CUDA cores, 2 = tensor-core MMA
int kvp_attn_d64(int variant, int G, const CUtensorMap *tmap, const kvp::AttnArgs *a, int P_req, int sm_count,
                 cudaStream_t st, int what, int *P_out);
int kvp_attn_d128(int variant, int G, const CUtensorMap *tmap, const kvp::AttnArgs *a, int P_req, int sm_count,
                  cudaStream_t st, int what, int *P_out);
int kvp_cascade_d64(int G, const CUtensorMap *tmap, const kvp::CascadeArgs *c, int grid, int sm_count,
                    cudaStream_t st, bool launch, int *P_out);
int kvp_cascade_d128(int G, const CUtensorMap *tmap, const kvp::CascadeArgs *c, int grid, int sm_count,
                     cudaStream_t st, bool launch, int *P_out);
