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

#include "pool_internal.h"

namespace {

// Fixed scratch for the split-K workspace.  It is device memory owned by this
// library's module: every GPU that loads the module holds it until the
// process exits.
constexpr size_t kScratchBytes = 32u << 20;  // 32 MiB

// Per-device address of the scratch array, resolved when a pool is created
// on the device (kvp_noalloc_prepare) or else on the first call.
constexpr int kMaxDevices = 64;
void *g_scratch_addr[kMaxDevices] = {};
std::mutex g_scratch_mu;

}  // namespace

// On the host this name is only a stand-in for the device array; its device
// address comes from cudaGetSymbolAddress.
static __device__ __align__(256) unsigned char g_attn_scratch[kScratchBytes];

namespace {

// Resolve the scratch address of device `dev`, which must be the current
// device (once per device).  The lookup loads the module that holds the
// array if it is not loaded yet (CUDA loads modules lazily by default), and
// that is when the array's 32 MiB are taken from the device.  On failure
// the runtime's last-error slot is cleared, so that the failure is not
// reported again by an unrelated later call on this thread.
int scratch_for_device(int dev, void **out)
{
    if (dev < 0 || dev >= kMaxDevices) return KV_ERR_UNSUPPORTED;
    std::lock_guard<std::mutex> g(g_scratch_mu);
    if (!g_scratch_addr[dev]) {
        void *p = nullptr;
        if (cudaGetSymbolAddress(&p, g_attn_scratch) != cudaSuccess || !p) {
            cudaGetLastError();
            return KV_ERR_CUDA;
        }
        g_scratch_addr[dev] = p;
    }
    *out = g_scratch_addr[dev];
    return KV_OK;
}

}  // namespace

// Called by kv_pool_create with the pool's device current: takes the
// scratch array's memory on that device before the caller fills the device
// with KV blocks, so a later first noalloc call needs no device memory.  A
// failure here is not an error of the pool; the first call retries.
void kvp_noalloc_prepare(int device)
{
    void *p = nullptr;
    (void)scratch_for_device(device, &p);
}

extern "C" {

int paged_decode_attn_noalloc(kv_pool *pool, int layout, const uint16_t *q, uint16_t *out,
                              const int32_t *dev_table, const int32_t *dev_ctx_lens, int max_blocks, int S,
                              int Hq, float scale, int num_splits, void *stream)
{
    size_t need = 0;
    int rc = kv_workspace_bytes(pool, layout, S, Hq, max_blocks, num_splits, &need);
    if (rc) return rc;
    if (need > kScratchBytes) return KV_ERR_WORKSPACE;  // batch too large for the fixed scratch
    // the scratch used must be the one on the pool's device, which is where
    // the kernels launch: the pool's device has to be the current one
    int dev = -1;
    if (cudaGetDevice(&dev) != cudaSuccess) {
        cudaGetLastError();
        return KV_ERR_CUDA;
    }
    if (dev != pool->device) return KV_ERR_INVALID_ARG;
    void *scratch = nullptr;
    rc = scratch_for_device(dev, &scratch);
    if (rc) return rc;
    return paged_decode_attn(pool, layout, q, out, dev_table, dev_ctx_lens, max_blocks, S, Hq, scale, num_splits,
                             scratch, kScratchBytes, stream);
}

}  // extern "C"
