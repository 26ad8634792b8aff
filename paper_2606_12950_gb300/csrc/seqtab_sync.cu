// seqtab_sync.cu -- kv_seqtab_sync: bring a device block table and length
// array up to date with a host sequence table.  Lengths and changed table
// entries travel as kernel parameters (no staging buffer, no per-row copy);
// a table whose changes exceed a quarter of it is copied whole.
#include <algorithm>

#include <cuda_runtime.h>

#include "seqtab_internal.h"
#include "stream_order.h"

namespace {

template <int WORDS>
struct SyncParams {
    int32_t *dev_table;
    int32_t *dev_lens;
    int32_t lens_begin;
    int32_t n_lens;
    int32_t n_patches;
    int32_t pad;
    int32_t data[WORDS];  // n_lens lengths, then n_patches (flat index, value) pairs
};

template <int WORDS>
__global__ void seqtab_sync_kernel(const __grid_constant__ SyncParams<WORDS> p)
{
    // a following programmatic-dependent grid may launch now; it waits for
    // this grid to complete before it reads the table or the lengths
    asm volatile("griddepcontrol.launch_dependents;" :::);
    // this grid is itself launched as a programmatic dependent (its launch
    // overlaps the previous kernel): wait for that kernel, which may still
    // read the lengths and the table, before writing them
    asm volatile("griddepcontrol.wait;" ::: "memory");
    for (int i = threadIdx.x; i < p.n_lens; i += blockDim.x) p.dev_lens[p.lens_begin + i] = p.data[i];
    for (int j = threadIdx.x; j < p.n_patches; j += blockDim.x)
        p.dev_table[p.data[p.n_lens + 2 * j]] = p.data[p.n_lens + 2 * j + 1];
}

// one launch carrying lens[li .. li + nl) and changed[pi .. pi + np)
template <int WORDS>
int launch_chunk(kv_seqtab *t, int32_t *dev_table, int32_t *dev_lens, size_t li, int nl, size_t pi, int np,
                 cudaStream_t st)
{
    SyncParams<WORDS> p;
    p.dev_table = dev_table;
    p.dev_lens = dev_lens;
    p.lens_begin = (int32_t)li;
    p.n_lens = nl;
    p.n_patches = np;
    p.pad = 0;
    for (int i = 0; i < nl; ++i) p.data[i] = t->lens[li + (size_t)i];
    for (int j = 0; j < np; ++j) {
        const int32_t idx = t->changed[pi + (size_t)j];
        p.data[nl + 2 * j] = idx;
        p.data[nl + 2 * j + 1] = t->table[(size_t)idx];
    }
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(1);
    cfg.blockDim = dim3(256);
    cfg.stream = st;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    if (cudaLaunchKernelEx(&cfg, seqtab_sync_kernel<WORDS>, p) != cudaSuccess) return KV_ERR_CUDA;
    kvp_note_stream(st, false);
    return KV_OK;
}

// parameter blocks of three sizes: a launch's cost grows with its parameter
// bytes, so a sync takes the smallest block that holds it
constexpr int kSmallWords = 256;
constexpr int kMidWords = 1016;    // about 4 KB of parameters
constexpr int kLargeWords = 4088;  // about 16 KB of parameters

}  // namespace

extern "C" int kv_seqtab_sync(kv_seqtab *t, int32_t *dev_table, int32_t *dev_ctx_lens, void *stream)
{
    if (!t || !dev_table || !dev_ctx_lens) return KV_ERR_INVALID_ARG;
    cudaStream_t st = (cudaStream_t)stream;
    const size_t total = (size_t)t->S * t->max_blocks;
    size_t np_all = t->changed.size();
    if (t->full_dirty || np_all * 4 > total) {
        // copy the whole table (pageable source: the call returns once the
        // runtime has staged it, so the host table may change afterwards)
        if (cudaMemcpyAsync(dev_table, t->table.data(), total * sizeof(int32_t), cudaMemcpyHostToDevice, st) !=
            cudaSuccess)
            return KV_ERR_CUDA;
        kvp_note_stream(st, false);
        t->counters.entries_uploaded += (int64_t)total;
        for (int32_t idx : t->changed) t->pending[(size_t)idx] = 0;
        t->changed.clear();
        t->full_dirty = false;
        np_all = 0;
    }
    size_t li = 0, pi = 0;
    const size_t S = (size_t)t->S;
    while (li < S || pi < np_all) {
        const size_t want = (S - li) + 2 * (np_all - pi);
        int rc;
        if (want <= (size_t)kSmallWords) {
            const int nl = (int)(S - li), np = (int)(np_all - pi);
            rc = launch_chunk<kSmallWords>(t, dev_table, dev_ctx_lens, li, nl, pi, np, st);
            li += (size_t)nl;
            pi += (size_t)np;
        } else if (want <= (size_t)kMidWords) {
            const int nl = (int)(S - li), np = (int)(np_all - pi);
            rc = launch_chunk<kMidWords>(t, dev_table, dev_ctx_lens, li, nl, pi, np, st);
            li += (size_t)nl;
            pi += (size_t)np;
        } else {
            const int nl = (int)std::min<size_t>(S - li, (size_t)kLargeWords);
            const int np = (int)std::min<size_t>(np_all - pi, (size_t)(kLargeWords - nl) / 2);
            rc = launch_chunk<kLargeWords>(t, dev_table, dev_ctx_lens, li, nl, pi, np, st);
            li += (size_t)nl;
            pi += (size_t)np;
        }
        if (rc) return rc;
        t->counters.sync_launches += 1;
    }
    t->counters.entries_uploaded += (int64_t)np_all;
    for (int32_t idx : t->changed) t->pending[(size_t)idx] = 0;
    t->changed.clear();
    return KV_OK;
}
