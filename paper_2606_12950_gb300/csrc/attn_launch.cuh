// attn_launch.cuh -- host-side launch of one paged-attention instantiation:
// stage count, shared memory, grid (one CTA per resident slot unless the
// caller asks for a given number of work partitions).
#pragma once

#include <algorithm>
#include <atomic>

#include "attn_impl.cuh"

namespace kvp {

// shared memory a CTA may use so that two CTAs fit on one SM
constexpr size_t kSmemBudget = 113 * 1024;

template <int D, int G, class Comp>
int attn_run(const CUtensorMap *tmap, AttnArgs a, int P_req, int sm_count, cudaStream_t st, bool launch,
             int *P_out)
{
    auto fn = paged_attn_kernel<D, G, Comp>;
    static std::atomic<bool> attr_set{false};
    if (!attr_set.load()) {
        if (cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, 227 * 1024) != cudaSuccess)
            return KV_ERR_CUDA;
        attr_set.store(true);
    }
    const size_t stage = 2ull * (D / 64) * kHalfBytes;
    const size_t fixed = attn_smem_bytes<D, G>(0, a.S);
    int nsw = 2;
    if (fixed < kSmemBudget) nsw = (int)std::min<size_t>(6, std::max<size_t>(2, (kSmemBudget - fixed) / (kWarps * stage)));
    const size_t smem = attn_smem_bytes<D, G>(nsw, a.S);
    if (smem > 227 * 1024) return KV_ERR_INVALID_ARG;
    int occ = 0;
    if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&occ, fn, kThreads, smem) != cudaSuccess) return KV_ERR_CUDA;
    const int P = P_req > 0 ? P_req : std::max(1, occ) * std::max(1, sm_count);
    *P_out = P;
    if (!launch) return KV_OK;
    a.nsw = nsw;
    a.P = P;
    fn<<<P, kThreads, smem, st>>>(*tmap, a);
    return cudaGetLastError() == cudaSuccess ? KV_OK : KV_ERR_CUDA;
}

}  // namespace kvp

// one entry per head dim; variant 1 = CUDA cores, 2 = tensor-core MMA
int kvp_attn_d64(int variant, int G, const CUtensorMap *tmap, const kvp::AttnArgs *a, int P_req, int sm_count,
                 cudaStream_t st, bool launch, int *P_out);
int kvp_attn_d128(int variant, int G, const CUtensorMap *tmap, const kvp::AttnArgs *a, int P_req, int sm_count,
                  cudaStream_t st, bool launch, int *P_out);
