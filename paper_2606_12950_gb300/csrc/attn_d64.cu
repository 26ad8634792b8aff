// attn_d64.cu -- instantiations of the paged decode attention kernel for
// head dim 64 (one translation unit per head dim keeps the build parallel).
#include "attn_launch.cuh"

int kvp_attn_d64(int variant, int G, const CUtensorMap *tmap, const kvp::AttnArgs *a, int P_req, int sm_count,
                 cudaStream_t st, int what, int *P_out)
{
    using namespace kvp;
#define KVP_CASE(GG)                                                                                   \
    case GG:                                                                                           \
        return variant == 1 ? attn_run<64, GG, FmaCompute<64, GG>>(tmap, *a, P_req, sm_count, st, what, P_out) \
                            : attn_run<64, GG, MmaCompute<64, GG>>(tmap, *a, P_req, sm_count, st, what, P_out);
    switch (G) {
        KVP_CASE(1)
        KVP_CASE(2)
        KVP_CASE(4)
        KVP_CASE(5)
    case 8:
        if (variant == 1) return KV_ERR_UNSUPPORTED;
        return attn_run<64, 8, MmaCompute<64, 8>>(tmap, *a, P_req, sm_count, st, what, P_out);
    default:
        return KV_ERR_UNSUPPORTED;
    }
#undef KVP_CASE
}

int kvp_cascade_d64(int G, const CUtensorMap *tmap, const kvp::CascadeArgs *c, int grid, int sm_count,
                    cudaStream_t st, bool launch, int *P_out)
{
    using namespace kvp;
    switch (G) {
    case 1: return cascade_run<64, 1>(tmap, c, grid, sm_count, st, launch, P_out);
    case 2: return cascade_run<64, 2>(tmap, c, grid, sm_count, st, launch, P_out);
    case 4: return cascade_run<64, 4>(tmap, c, grid, sm_count, st, launch, P_out);
    case 5: return cascade_run<64, 5>(tmap, c, grid, sm_count, st, launch, P_out);
    case 8: return cascade_run<64, 8>(tmap, c, grid, sm_count, st, launch, P_out);
    default: return KV_ERR_UNSUPPORTED;
    }
}
