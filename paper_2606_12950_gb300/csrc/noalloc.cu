// noalloc.cu -- paged decode attention for callers that cannot allocate.
//
// paged_decode_attn needs a device workspace (the split index and the fp32
// split partials), which the caller normally allocates.  Some callers cannot
// do that: a serving loop that has handed all free device memory to the KV
// pool, a framework whose allocator this layer may not call, or a decode
// loop where a cudaMalloc (which can synchronise the whole device) is not
// acceptable.  paged_decode_attn_noalloc serves them with a fixed scratch
// array that lives in this file, so the call allocates nothing.
#include <mutex>

#include <cuda_runtime.h>

#include "kvpool.h"

namespace {

// Fixed scratch for the split-K workspace.  It is device memory owned by this
// library's module: every GPU that loads the module holds it until the
// process exits.
constexpr size_t kScratchBytes = 32u << 20;  // 32 MiB

// Per-device address of the scratch array, resolved on first use.
constexpr int kMaxDevices = 64;
void *g_scratch_addr[kMaxDevices] = {};
std::mutex g_scratch_mu;

}  // namespace

// On the host this name is only a stand-in for the device array; its device
// address comes from cudaGetSymbolAddress.
static __device__ __align__(256) unsigned char g_attn_scratch[kScratchBytes];

namespace {

// Resolve the scratch address for the current device (once per device).
int scratch_for_current_device(void **out)
{
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) return KV_ERR_CUDA;
    if (dev < 0 || dev >= kMaxDevices) return KV_ERR_UNSUPPORTED;
    std::lock_guard<std::mutex> g(g_scratch_mu);
    if (!g_scratch_addr[dev]) {
        void *p = nullptr;
        if (cudaGetSymbolAddress(&p, g_attn_scratch) != cudaSuccess || !p) return KV_ERR_CUDA;
        g_scratch_addr[dev] = p;
    }
    *out = g_scratch_addr[dev];
    return KV_OK;
}

}  // namespace

extern "C" {

int paged_decode_attn_noalloc(kv_pool *pool, int layout, const uint16_t *q, uint16_t *out,
                              const int32_t *dev_table, const int32_t *dev_ctx_lens, int max_blocks, int S,
                              int Hq, float scale, int num_splits, void *stream)
{
    size_t need = 0;
    int rc = kv_workspace_bytes(pool, layout, S, Hq, max_blocks, num_splits, &need);
    if (rc) return rc;
    if (need > kScratchBytes) return KV_ERR_WORKSPACE;  // batch too large for the fixed scratch
    void *scratch = nullptr;
    rc = scratch_for_current_device(&scratch);
    if (rc) return rc;
    return paged_decode_attn(pool, layout, q, out, dev_table, dev_ctx_lens, max_blocks, S, Hq, scale, num_splits,
                             scratch, kScratchBytes, stream);
}

}  // extern "C"
