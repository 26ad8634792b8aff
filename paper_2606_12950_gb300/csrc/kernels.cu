// kernels.cu -- KV append kernel, the shared-prefix plan kernel and the
// launch wrappers of the C ABI: kv_append, kv_workspace_bytes,
// kv_cascade_workspace_bytes, paged_decode_attn(_append), the table sync
// carried by the decode launch (paged_decode_attn_seqtab), co-located
// batches as one chain (paged_decode_attn_multi) and shared-prefix
// attention (paged_decode_attn_cascade).
#include <algorithm>
#include <atomic>
#include <chrono>
#include <cmath>
#include <memory>
#include <mutex>
#include <vector>

#include <cudaTypedefs.h>
#include <cuda_runtime.h>

#include "attn_launch.cuh"
#include "pool_internal.h"
#include "seqtab_internal.h"

// ---- stream_order.h: the library's latest launch per stream.  A small table
// (streams in use at once are few); a stream that fell out of it reads as
// "not after a combine", the safe answer.
namespace {
constexpr int kStreamSlots = 64;
struct StreamNote {
    void *stream;
    bool combine;
    uint64_t stamp;
    KvpCascadeNote cascade;  // ws null: not a shared-prefix combine
};
std::mutex g_stream_mu;
StreamNote g_streams[kStreamSlots];
uint64_t g_stream_clock = 0;
}  // namespace

void kvp_note_stream(void *stream, bool combine)
{
    std::lock_guard<std::mutex> lk(g_stream_mu);
    int slot = -1, oldest = 0;
    for (int i = 0; i < kStreamSlots; ++i) {
        if (g_streams[i].stamp && g_streams[i].stream == stream) {
            slot = i;
            break;
        }
        if (g_streams[i].stamp < g_streams[oldest].stamp) oldest = i;
    }
    if (slot < 0) slot = oldest;
    g_streams[slot] = StreamNote{stream, combine, ++g_stream_clock, KvpCascadeNote{}};
}

void kvp_note_cascade_combine(void *stream, const KvpCascadeNote &n)
{
    std::lock_guard<std::mutex> lk(g_stream_mu);
    for (int i = 0; i < kStreamSlots; ++i)
        if (g_streams[i].stamp && g_streams[i].stream == stream && g_streams[i].combine) g_streams[i].cascade = n;
}

bool kvp_stream_after_cascade(void *stream, KvpCascadeNote *n)
{
    std::lock_guard<std::mutex> lk(g_stream_mu);
    for (int i = 0; i < kStreamSlots; ++i)
        if (g_streams[i].stamp && g_streams[i].stream == stream) {
            if (!g_streams[i].combine || !g_streams[i].cascade.ws) return false;
            *n = g_streams[i].cascade;
            return true;
        }
    return false;
}

bool kvp_stream_after_combine(void *stream)
{
    std::lock_guard<std::mutex> lk(g_stream_mu);
    for (int i = 0; i < kStreamSlots; ++i)
        if (g_streams[i].stamp && g_streams[i].stream == stream) return g_streams[i].combine;
    return false;
}

namespace {

// Append: the decode step writes the new token's K and V before attending
// (§II).  One thread per 16-byte chunk of a (sequence, KV head, K|V) row; 16
// consecutive threads write one 256-byte row (d = 128), so stores coalesce.
__global__ void append_kernel(uint8_t *__restrict__ pool, const uint4 *__restrict__ k_new,
                              const uint4 *__restrict__ v_new, const int32_t *__restrict__ table,
                              const int32_t *__restrict__ ctx_lens, int32_t *err, int S, int Hkv, int D, int bs,
                              int max_blocks, int64_t page_bytes, int64_t n_pages, int32_t pages_per_block)
{
    const int cpr = D / 8;  // 16-byte chunks per row
    const int64_t total = (int64_t)S * Hkv * 2 * cpr;
    for (int64_t idx = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; idx < total;
         idx += (int64_t)gridDim.x * blockDim.x) {
        const int c = (int)(idx % cpr);
        int64_t rest = idx / cpr;
        const int kv = (int)(rest % 2);
        rest /= 2;
        const int g = (int)(rest % Hkv);
        const int s = (int)(rest / Hkv);
        const int32_t n = ctx_lens[s];
        if (n <= 0) continue;
        if (n > max_blocks * bs) {
            atomicCAS(err, 0, KV_ERR_DEVICE_BOUNDS);
            continue;
        }
        const int pos = n - 1;
        const int32_t phys = table[(int64_t)s * max_blocks + pos / bs];
        if (phys < 0 || (int64_t)phys + pages_per_block > n_pages) {
            atomicCAS(err, 0, KV_ERR_DEVICE_BOUNDS);
            continue;
        }
        const uint4 *src = (kv ? v_new : k_new) + ((int64_t)s * Hkv + g) * cpr + c;
        uint8_t *dst = pool + (int64_t)phys * page_bytes +
                       ((((int64_t)kv * Hkv + g) * bs + (pos % bs)) * D + (int64_t)c * 8) * 2;
        *reinterpret_cast<uint4 *>(dst) = *src;
    }
}

PFN_cuTensorMapEncodeTiled_v12000 encode_fn()
{
    static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
    static std::once_flag once;
    std::call_once(once, [] {
        void *p = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) ==
                cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(p);
    });
    return fn;
}

// The pool seen as a 2-D bf16 tensor of rows of d elements; a box is 64
// columns x 16 rows with the 128-byte swizzle, i.e. one half of a 16-token
// K or V tile of one head.
int ensure_tmap(kv_pool *p, int layout)
{
    std::lock_guard<std::mutex> g(p->mu);
    if (p->tmap_ok[layout]) return KV_OK;
    auto enc = encode_fn();
    if (!enc) return KV_ERR_CUDA;
    const int D = p->desc.layouts[layout].head_dim;
    const uint64_t rows = (uint64_t)p->n_pages * p->page_bytes / ((uint64_t)D * 2);
    cuuint64_t dims[2] = {(cuuint64_t)D, (cuuint64_t)rows};
    cuuint64_t strides[1] = {(cuuint64_t)D * 2};
    cuuint32_t box[2] = {64, (cuuint32_t)kvp::kTile};
    cuuint32_t estr[2] = {1, 1};
    CUresult r = enc(&p->tmap[layout], CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, p->desc.device_base, dims, strides, box,
                     estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                     CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    if (r != CUDA_SUCCESS) return KV_ERR_CUDA;
    p->tmap_ok[layout] = true;
    return KV_OK;
}

bool aligned16(const void *ptr) { return ((uintptr_t)ptr & 15u) == 0; }

int pick_variant(const kv_pool *p, int G)
{
    if (p->attn_variant) return p->attn_variant;
    (void)G;
    return 2;
}

// common argument checks of paged_decode_attn / kv_workspace_bytes
int attn_shape(const kv_pool *p, int layout, int S, int Hq, int max_blocks, int *G_out)
{
    if (!p || layout < 0 || layout >= p->desc.num_layouts) return KV_ERR_INVALID_ARG;
    if (S < 0 || max_blocks < 1 || Hq < 1) return KV_ERR_INVALID_ARG;
    const kv_layout &L = p->desc.layouts[layout];
    if (Hq % L.num_kv_heads) return KV_ERR_INVALID_ARG;
    const int G = Hq / L.num_kv_heads;
    if (L.head_dim != 64 && L.head_dim != 128) return KV_ERR_UNSUPPORTED;
    if (p->desc.block_size % kvp::kTile) return KV_ERR_UNSUPPORTED;
    if (!(G == 1 || G == 2 || G == 4 || G == 5 || G == 8)) return KV_ERR_UNSUPPORTED;
    // unit ids and pool rows are 32-bit on the device
    const int64_t tiles = ((int64_t)max_blocks * p->desc.block_size + kvp::kTile - 1) / kvp::kTile;
    if ((int64_t)S * tiles * L.num_kv_heads >= INT32_MAX) return KV_ERR_INVALID_ARG;
    if ((int64_t)p->n_pages * (int64_t)p->page_bytes / (2 * L.head_dim) >= INT32_MAX) return KV_ERR_INVALID_ARG;
    if ((int64_t)max_blocks * p->desc.block_size >= INT32_MAX) return KV_ERR_INVALID_ARG;
    *G_out = G;
    return KV_OK;
}

int dispatch(int variant, int D, int G, const CUtensorMap *tmap, const kvp::AttnArgs *a, int P_req, int sms,
             cudaStream_t st, int what, int *P_out)
{
    if (D == 64) return kvp_attn_d64(variant, G, tmap, a, P_req, sms, st, what, P_out);
    return kvp_attn_d128(variant, G, tmap, a, P_req, sms, st, what, P_out);
}

// a host sequence table whose pending changes travel with a launch (the
// decode launch, or the plan kernel's in shared-prefix mode)
struct FusedSync {
    kv_seqtab *t;
    int32_t *dev_table;
    int32_t *dev_lens;
};

// The shared-prefix plan, carried as this kernel's parameters, into the
// workspace: the whole plan for the prefix kernel, and the per-sequence
// skips (its last S words) where the decode kernel (suffix tiles start
// there) and the combine read them; with a fused table sync also a
// sequence table's lengths and changed entries, into the device lengths
// and table (what the sync kernel would write), which saves that kernel's
// launch and its grid-to-grid hand-off.  It waits for the previous grid
// first: the previous step's kernels may still read the old plan, skips,
// lengths and table.  The parameter block comes in three sizes so that a
// small plan does not pay for copying the largest one into every launch
// (host and device time).
template <int W>
struct PlanParams {
    int32_t *ws_plan;
    int32_t *ws_skip;
    int32_t *sync_table;  // fused table sync: null for none
    int32_t *sync_lens;
    uint64_t *flags;      // overlap: [0] set to epoch once everything is written, [1] once the grids before completed
    uint64_t epoch;
    int32_t overlap;
    int32_t n_words;      // plan words
    int32_t S;
    int32_t sync_nlens;
    int32_t sync_npatch;
    int32_t words[W];  // the plan, then sync_nlens lengths, then sync_npatch (flat index, value) pairs
};

template <int W>
__global__ void cascade_plan_kernel(const __grid_constant__ PlanParams<W> p)
{
    // Alone: the grids before (the previous step's kernels, which read the
    // plan, the skips, the lengths and the table) have completed after this
    // wait; the grid after waits for this one to complete before it reads
    // any of them.  Overlapping the previous step's shared-prefix combine
    // (overlap): that combine reads none of what is written here (its skips
    // are the other of the workspace's two skip arrays), so everything is
    // written at once and flags[0] tells the decode grid, which does not
    // wait for this grid; flags[1] tells it when the combine has completed.
    // The prefix grid still waits for this grid to complete, which is after
    // the wait below.
    if (!p.overlap) kvp::grid_dependency_wait();
    kvp::grid_launch_dependents();
    for (int i = threadIdx.x; i < p.n_words; i += blockDim.x) p.ws_plan[i] = p.words[i];
    const int32_t *skip = p.words + (p.n_words - p.S);
    for (int s = threadIdx.x; s < p.S; s += blockDim.x) p.ws_skip[s] = skip[s];
    if (p.sync_table) {
        const int32_t *lw = p.words + p.n_words, *pw = lw + p.sync_nlens;
        for (int i = threadIdx.x; i < p.sync_nlens; i += blockDim.x) p.sync_lens[i] = lw[i];
        for (int j = threadIdx.x; j < p.sync_npatch; j += blockDim.x) p.sync_table[pw[2 * j]] = pw[2 * j + 1];
    }
    if (!p.overlap) return;
    __syncthreads();
    if (threadIdx.x == 0) {
        __threadfence();
        kvp::st_release_gpu(p.flags, p.epoch);
        kvp::grid_dependency_wait();
        kvp::st_release_gpu(p.flags + 1, p.epoch);
    }
}

// a plan launch that overlaps the previous step's shared-prefix combine
struct PlanOverlap {
    bool on;
    uint64_t *flags;
    uint64_t epoch;
};

// A fresh 64-bit tag per overlapping call: the decode kernel takes a flag
// as set only when it holds this call's tag, so a flag left by an earlier
// call, or whatever the workspace held before, is never taken for it.
// SplitMix64 (Steele, Lea and Flood, 2014) over a counter, salted per
// process.
uint64_t next_epoch()
{
    static std::atomic<uint64_t> ctr{0};
    static const uint64_t salt =
        (uint64_t)std::chrono::steady_clock::now().time_since_epoch().count() ^ (uint64_t)(uintptr_t)&ctr;
    uint64_t z = salt + 0x9E3779B97F4A7C15ull * (ctr.fetch_add(1, std::memory_order_relaxed) + 1);
    z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
    z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
    z ^= z >> 31;
    return z ? z : 1;
}

// parameter blocks of three sizes (a launch's host cost grows with its
// parameter bytes): about 4, 8 and 16 KB
constexpr int kPlanSmallWords = 1024;
constexpr int kPlanMidWords = 2040;

template <int W>
int cascade_plan_launch(const int32_t *words, int n_words, int S, int32_t *ws_plan, int32_t *ws_skip,
                        const FusedSync *sync, const PlanOverlap &ov, cudaStream_t st)
{
    static thread_local std::unique_ptr<PlanParams<W>> buf(new PlanParams<W>());
    PlanParams<W> *p = buf.get();
    p->ws_plan = ws_plan;
    p->ws_skip = ws_skip;
    p->flags = ov.flags;
    p->epoch = ov.epoch;
    p->overlap = ov.on ? 1 : 0;
    p->n_words = n_words;
    p->S = S;
    std::copy(words, words + n_words, p->words);
    p->sync_table = nullptr;
    p->sync_lens = nullptr;
    p->sync_nlens = 0;
    p->sync_npatch = 0;
    if (sync) {
        const kv_seqtab *t = sync->t;
        const int nl = t->S, np = (int)t->changed.size();
        int32_t *w = p->words + n_words;
        for (int i = 0; i < nl; ++i) w[i] = t->lens[(size_t)i];
        for (int j = 0; j < np; ++j) {
            const int32_t idx = t->changed[(size_t)j];
            w[nl + 2 * j] = idx;
            w[nl + 2 * j + 1] = t->table[(size_t)idx];
        }
        p->sync_table = sync->dev_table;
        p->sync_lens = sync->dev_lens;
        p->sync_nlens = nl;
        p->sync_npatch = np;
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
    if (cudaLaunchKernelEx(&cfg, cascade_plan_kernel<W>, *p) != cudaSuccess) return KV_ERR_CUDA;
    kvp_note_stream(st, false);
    return KV_OK;
}

// words the plan kernel carries: the plan's, plus the sync's lengths and
// changed entries when it is fused
inline size_t plan_sync_words(int n_words, const FusedSync *sync)
{
    return (size_t)n_words + (sync ? (size_t)sync->t->S + 2 * sync->t->changed.size() : 0);
}

int cascade_plan_run(const int32_t *words, int n_words, int S, int32_t *ws_plan, int32_t *ws_skip,
                     const FusedSync *sync, const PlanOverlap &ov, cudaStream_t st)
{
    const size_t n = plan_sync_words(n_words, sync);
    if (n <= (size_t)kPlanSmallWords)
        return cascade_plan_launch<kPlanSmallWords>(words, n_words, S, ws_plan, ws_skip, sync, ov, st);
    if (n <= (size_t)kPlanMidWords)
        return cascade_plan_launch<kPlanMidWords>(words, n_words, S, ws_plan, ws_skip, sync, ov, st);
    if (n > (size_t)kvp::kCascadeWords) return KV_ERR_INVALID_ARG;  // the caller syncs separately first
    return cascade_plan_launch<kvp::kCascadeWords>(words, n_words, S, ws_plan, ws_skip, sync, ov, st);
}

// workspace: per-run (first part, parts) as int2 (padded to 256 bytes),
// then the fp32 partials
size_t ws_layout(int S, int Hkv, int G, int D, int P, size_t *part_off)
{
    const size_t hdr = ((size_t)S * Hkv * sizeof(int2) + 255) / 256 * 256;
    *part_off = hdr;
    return hdr + kvp::attn_partial_slots(S, Hkv, P) * (size_t)((G * D + 2 * G + 3) / 4 * 4) * 4;
}

// cascade workspace: the above, then two arrays of per-sequence skips (each
// padded to 256 bytes; consecutive calls use different ones, so that a plan
// kernel can write its skips while the previous step's combine still reads
// the other), the plan kernel's two flags (256 bytes), the plan words
// (kCascadeWords, padded), then kMaxKeySplits prefix records per (sequence,
// KV head)
size_t cascade_ws_layout(int S, int Hkv, int G, int D, int P, size_t *part_off, size_t *skip_off, size_t *pre_off,
                         size_t *plan_off, size_t *flags_off = nullptr)
{
    const size_t base = (ws_layout(S, Hkv, G, D, P, part_off) + 255) / 256 * 256;
    const size_t skip_bytes = ((size_t)S * 4 + 255) / 256 * 256;
    *skip_off = base;
    if (flags_off) *flags_off = base + 2 * skip_bytes;
    *plan_off = base + 2 * skip_bytes + 256;
    *pre_off = *plan_off + ((size_t)kvp::kCascadeWords * 4 + 255) / 256 * 256;
    return *pre_off + (size_t)kvp::kMaxKeySplits * S * Hkv * (size_t)((G * D + 2 * G + 3) / 4 * 4) * 4;
}

int cascade_dispatch(int D, int G, const CUtensorMap *tmap, const kvp::CascadeArgs *c, int grid, int sms,
                     cudaStream_t st, bool launch, int *P_out)
{
    if (D == 64) return kvp_cascade_d64(G, tmap, c, grid, sms, st, launch, P_out);
    return kvp_cascade_d128(G, tmap, c, grid, sms, st, launch, P_out);
}

}  // namespace

extern "C" {

int kv_append(kv_pool *p, int layout, const uint16_t *k_new, const uint16_t *v_new, const int32_t *dev_table,
              const int32_t *dev_ctx_lens, int max_blocks, int S, void *stream)
{
    if (!p || layout < 0 || layout >= p->desc.num_layouts || S < 0 || max_blocks < 1) return KV_ERR_INVALID_ARG;
    if (S == 0) return KV_OK;
    if (!k_new || !v_new || !dev_table || !dev_ctx_lens) return KV_ERR_INVALID_ARG;
    if (!aligned16(k_new) || !aligned16(v_new)) return KV_ERR_INVALID_ARG;
    const kv_layout &L = p->desc.layouts[layout];
    if (L.head_dim % 8) return KV_ERR_UNSUPPORTED;
    const int64_t total = (int64_t)S * L.num_kv_heads * 2 * (L.head_dim / 8);
    const int threads = 256;
    const int64_t want = (total + threads - 1) / threads;
    const int blocks = (int)std::min<int64_t>(want, (int64_t)std::max(1, p->sm_count) * 16);
    append_kernel<<<blocks, threads, 0, (cudaStream_t)stream>>>(
        (uint8_t *)p->desc.device_base, reinterpret_cast<const uint4 *>(k_new), reinterpret_cast<const uint4 *>(v_new),
        dev_table, dev_ctx_lens, p->desc.device_error, S, L.num_kv_heads, L.head_dim, p->desc.block_size, max_blocks,
        (int64_t)p->page_bytes, p->n_pages, p->pages_per_block[layout]);
    kvp_note_stream(stream, false);
    return cudaGetLastError() == cudaSuccess ? KV_OK : KV_ERR_CUDA;
}

int kv_workspace_bytes(const kv_pool *p, int layout, int S, int Hq, int max_blocks, int num_splits,
                       size_t *out_bytes)
{
    int G = 0;
    if (!out_bytes || num_splits < 0) return KV_ERR_INVALID_ARG;
    int rc = attn_shape(p, layout, S, Hq, max_blocks, &G);
    if (rc) return rc;
    const kv_layout &L = p->desc.layouts[layout];
    kvp::AttnArgs a{};
    a.S = S;
    a.Hkv = L.num_kv_heads;
    int P = 0;
    rc = dispatch(pick_variant(p, G), L.head_dim, G, nullptr, &a, num_splits, p->sm_count, nullptr, kvp::kLaunchQuery, &P);
    if (rc) return rc;
    size_t off;
    *out_bytes = ws_layout(S, L.num_kv_heads, G, L.head_dim, P, &off);
    return KV_OK;
}

int kv_cascade_workspace_bytes(const kv_pool *p, int layout, int S, int Hq, int max_blocks, size_t *out_bytes)
{
    int G = 0;
    if (!out_bytes) return KV_ERR_INVALID_ARG;
    int rc = attn_shape(p, layout, S, Hq, max_blocks, &G);
    if (rc) return rc;
    const kv_layout &L = p->desc.layouts[layout];
    kvp::AttnArgs a{};
    a.S = S;
    a.Hkv = L.num_kv_heads;
    int P = 0;
    rc = dispatch(pick_variant(p, G), L.head_dim, G, nullptr, &a, 0, p->sm_count, nullptr, kvp::kLaunchQuery, &P);
    if (rc) return rc;
    size_t o1, o2, o3, o4;
    *out_bytes = cascade_ws_layout(S, L.num_kv_heads, G, L.head_dim, P, &o1, &o2, &o3, &o4);
    return KV_OK;
}

}  // extern "C"

namespace {

struct CascadePlan {
    const kv_prefix_group *groups;
    int n_groups;
    const int32_t *members;
};

int attn_call(kv_pool *p, int layout, const uint16_t *q, const uint16_t *k_new, const uint16_t *v_new,
              uint16_t *out, const int32_t *dev_table, const int32_t *dev_ctx_lens, int max_blocks, int S, int Hq,
              float scale, int num_splits, void *workspace, size_t ws_bytes, void *stream,
              const CascadePlan *cas = nullptr, const FusedSync *sync = nullptr)
{
    int G = 0;
    if (num_splits < 0 || !std::isfinite(scale)) return KV_ERR_INVALID_ARG;
    int rc = attn_shape(p, layout, S, Hq, max_blocks, &G);
    if (rc) return rc;
    if (S == 0) return KV_OK;
    if (!q || !out || !dev_table || !dev_ctx_lens || !aligned16(q) || !aligned16(out)) return KV_ERR_INVALID_ARG;
    if ((k_new || v_new) && (!k_new || !v_new || !aligned16(k_new) || !aligned16(v_new))) return KV_ERR_INVALID_ARG;
    if (p->sm_count <= 0) return KV_ERR_CUDA;
    const kv_layout &L = p->desc.layouts[layout];
    const int variant = pick_variant(p, G);
    kvp::AttnArgs a{};
    a.q = q;
    a.out = out;
    a.k_new = k_new;
    a.v_new = v_new;
    a.pool = reinterpret_cast<uint16_t *>(p->desc.device_base);
    a.table = dev_table;
    a.ctx_lens = dev_ctx_lens;
    a.err = p->desc.device_error;
    a.rows_per_page = (int64_t)(p->page_bytes / (2ull * L.head_dim));
    a.pool_pages = p->n_pages;
    a.pages_per_block = p->pages_per_block[layout];
    a.max_blocks = max_blocks;
    a.S = S;
    a.Hkv = L.num_kv_heads;
    a.bs = p->desc.block_size;
    a.qk_scale = scale * 1.4426950408889634f;
    int P = 0;
    rc = dispatch(variant, L.head_dim, G, nullptr, &a, num_splits, p->sm_count, nullptr, kvp::kLaunchQuery, &P);
    if (rc) return rc;
    size_t part_off;
    if (!cas) {
        const size_t need = ws_layout(S, L.num_kv_heads, G, L.head_dim, P, &part_off);
        if (!workspace || ws_bytes < need || ((uintptr_t)workspace & 255u)) return KV_ERR_WORKSPACE;
        a.ws_run = reinterpret_cast<int2 *>(workspace);
        a.ws_part = reinterpret_cast<float *>(reinterpret_cast<uint8_t *>(workspace) + part_off);
        rc = ensure_tmap(p, layout);
        if (rc) return rc;
        if (sync) {
            // the caller checked that the lengths and changed entries fit
            kv_seqtab *t = sync->t;
            const int nl = t->S, np = (int)t->changed.size();
            a.sync_table = sync->dev_table;
            a.sync_lens = sync->dev_lens;
            a.sync_nlens = nl;
            a.sync_npatch = np;
            for (int i = 0; i < nl; ++i) a.sync_words[i] = t->lens[(size_t)i];
            for (int j = 0; j < np; ++j) {
                const int32_t idx = t->changed[(size_t)j];
                a.sync_words[nl + 2 * j] = idx;
                a.sync_words[nl + 2 * j + 1] = t->table[(size_t)idx];
            }
        }
        // right after one of this library's combines on the stream, and with
        // the pool's step overlap on, the decode grid starts while that
        // combine finishes (chain 3)
        const bool overlap = p->step_overlap && kvp_stream_after_combine(stream);
        if (overlap) a.chain = 3;
        rc = dispatch(variant, L.head_dim, G, &p->tmap[layout], &a, num_splits, p->sm_count, (cudaStream_t)stream,
                      kvp::kLaunchBoth, &P);
        if (rc == KV_OK && overlap) p->overlapped.fetch_add(1, std::memory_order_relaxed);
        if (rc || !sync) return rc;
        kv_seqtab *t = sync->t;
        t->counters.entries_uploaded += (int64_t)t->changed.size();
        for (int32_t idx : t->changed) t->pending[(size_t)idx] = 0;
        t->changed.clear();
        return KV_OK;
    }

    // ---- shared-prefix mode: validate the plan and build the prefix
    // kernel's parameters, then launch, in stream order: the plan kernel
    // (per-sequence skips), the prefix kernel, the decode kernel over the
    // suffixes and the combine.  The prefix kernel takes about a quarter of
    // the SMs (one CTA each); the decode kernel, sized to the SMs left, runs
    // beside it without waiting for it and waits for it at its end, so the
    // combine, which waits for the decode grid, sees both grids' records ----
    const int bs = p->desc.block_size, Hkv = L.num_kv_heads;
    const int ng = cas->n_groups;
    if (ng < 1 || !cas->groups || !cas->members) return KV_ERR_INVALID_ARG;
    int64_t nm = 0;
    for (int i = 0; i < ng; ++i) {
        const kv_prefix_group &gr = cas->groups[i];
        if (gr.count < 1 || gr.tokens < kvp::kPreChunk || gr.tokens % kvp::kPreChunk || gr.tokens % bs ||
            (int64_t)gr.tokens > (int64_t)max_blocks * bs)
            return KV_ERR_INVALID_ARG;
        nm += gr.count;
    }
    if (nm > S || 2 * (ng + 1) + ng + nm + S > kvp::kCascadeWords) return KV_ERR_INVALID_ARG;
    // the plan's words are built in a per-thread buffer; the plan kernel
    // carries them to the workspace
    static thread_local std::vector<int32_t> words_buf;
    const int n_words = (int)(2 * (ng + 1) + ng + nm + S);
    words_buf.resize((size_t)n_words);
    kvp::CascadeArgs cargs{};
    kvp::CascadeArgs *c = &cargs;
    int32_t *tile_off = words_buf.data(), *mem_off = tile_off + ng + 1, *tokens = mem_off + ng + 1;
    int32_t *mem = tokens + ng, *skip = mem + nm;
    std::fill(skip, skip + S, 0);
    const int MT = kvp::kPreQTiles * (kvp::kPreRows / G);  // members per prefix CTA
    int kt_min = INT32_MAX;
    tile_off[0] = 0;
    mem_off[0] = 0;
    for (int i = 0; i < ng; ++i) {
        const kv_prefix_group &gr = cas->groups[i];
        tile_off[i + 1] = tile_off[i] + (gr.count + MT - 1) / MT;
        mem_off[i + 1] = mem_off[i] + gr.count;
        tokens[i] = gr.tokens;
        kt_min = std::min(kt_min, gr.tokens / kvp::kPreChunk);
        for (int j = mem_off[i]; j < mem_off[i + 1]; ++j) {
            const int32_t s = cas->members[j];
            if (s < 0 || s >= S || skip[s]) return KV_ERR_INVALID_ARG;  // each sequence in one group at most
            mem[j] = s;
            skip[s] = gr.tokens;
        }
    }
    const int tiles = tile_off[ng];
    size_t skip_off, pre_off, plan_off, flags_off;
    const size_t need =
        cascade_ws_layout(S, Hkv, G, L.head_dim, P, &part_off, &skip_off, &pre_off, &plan_off, &flags_off);
    if (!workspace || ws_bytes < need || ((uintptr_t)workspace & 255u)) return KV_ERR_WORKSPACE;
    uint8_t *ws = reinterpret_cast<uint8_t *>(workspace);
    c->q = q;
    c->table = dev_table;
    c->err = p->desc.device_error;
    c->ws_pre = reinterpret_cast<float *>(ws + pre_off);
    c->ws_skip = reinterpret_cast<int32_t *>(ws + skip_off);
    c->plan = reinterpret_cast<const int32_t *>(ws + plan_off);
    c->rows_per_page = a.rows_per_page;
    c->pool_pages = a.pool_pages;
    c->pages_per_block = a.pages_per_block;
    c->max_blocks = max_blocks;
    c->S = S;
    c->Hkv = Hkv;
    c->bs = bs;
    c->n_groups = ng;
    c->n_members = (int32_t)nm;
    c->qk_scale = a.qk_scale;
    int P_pre = 0;
    rc = cascade_dispatch(L.head_dim, G, nullptr, c, 0, p->sm_count, nullptr, false, &P_pre);
    if (rc) return rc;
    // key splits: as many as keep the prefix grid within a quarter of the
    // GPU's CTA slots for it (at least one; every split non-empty)
    const int pre_slots = std::max(1, P_pre / 4);
    c->KS = std::max(1, std::min({pre_slots / std::max(1, tiles * Hkv), kvp::kMaxKeySplits, kt_min}));
    // the decode grid fills the SMs the prefix grid leaves free (all of them
    // when the prefix grid needs more than half the GPU: the decode CTAs then
    // start as prefix CTAs finish)
    const int pre_ctas = tiles * Hkv * c->KS;
    const int pre_occ = std::max(1, P_pre / std::max(1, p->sm_count));
    const int pre_sms = (pre_ctas + pre_occ - 1) / pre_occ;
    const int free_sms = 2 * pre_sms <= p->sm_count ? p->sm_count - pre_sms : p->sm_count;
    if (num_splits <= 0) {
        rc = dispatch(variant, L.head_dim, G, nullptr, &a, 0, free_sms, nullptr, kvp::kLaunchQuery, &P);
        if (rc) return rc;
        num_splits = P;
    }
    a.ws_run = reinterpret_cast<int2 *>(ws);
    a.ws_part = reinterpret_cast<float *>(ws + part_off);
    a.chain = 2;  // beside the prefix kernel, which waits before releasing it
    a.ws_pre = c->ws_pre;
    a.KS = c->KS;
    rc = ensure_tmap(p, layout);
    if (rc) return rc;
    // a table sync that does not fit the plan kernel's parameters (or a
    // table never written to the device) runs as its own launches first
    if (sync && (sync->t->full_dirty || plan_sync_words(n_words, sync) > (size_t)kvp::kCascadeWords)) {
        rc = kv_seqtab_sync(sync->t, sync->dev_table, sync->dev_lens, stream);
        if (rc) return rc;
        sync = nullptr;
    }
    // The skips go to the skip array the previous call on this workspace did
    // not use.  Right after that call's combine (same workspace and layout),
    // with the pool's step overlap on, this step overlaps the combine: the
    // plan kernel writes at once and raises its flags, the prefix kernel
    // releases the decode kernel before its wait, and the decode kernel
    // (chain 4) reads after the first flag and writes after the second.
    int32_t *skip0 = reinterpret_cast<int32_t *>(ws + skip_off);
    int32_t *skip1 = reinterpret_cast<int32_t *>(ws + skip_off + ((size_t)S * 4 + 255) / 256 * 256);
    uint64_t *flags = reinterpret_cast<uint64_t *>(ws + flags_off);
    KvpCascadeNote prev{};
    const bool same_ws = kvp_stream_after_cascade(stream, &prev) && prev.ws == workspace && prev.flags == flags &&
                         prev.plan == ws + plan_off && (prev.skip == skip0 || prev.skip == skip1);
    c->ws_skip = same_ws && prev.skip == skip0 ? skip1 : skip0;
    a.skip = c->ws_skip;
    PlanOverlap ov{p->step_overlap && same_ws, flags, 0};
    if (ov.on) {
        ov.epoch = next_epoch();
        a.chain = 4;
        a.flags = flags;
        a.epoch = ov.epoch;
    }
    c->overlap = ov.on ? 1 : 0;
    rc = cascade_plan_run(words_buf.data(), n_words, S, reinterpret_cast<int32_t *>(ws + plan_off), c->ws_skip,
                          sync, ov, (cudaStream_t)stream);
    if (rc) return rc;
    if (sync) {
        kv_seqtab *t = sync->t;
        t->counters.entries_uploaded += (int64_t)t->changed.size();
        for (int32_t idx : t->changed) t->pending[(size_t)idx] = 0;
        t->changed.clear();
    }
    rc = cascade_dispatch(L.head_dim, G, &p->tmap[layout], c, pre_ctas, p->sm_count, (cudaStream_t)stream, true,
                          &P_pre);
    if (rc) return rc;
    rc = dispatch(variant, L.head_dim, G, &p->tmap[layout], &a, num_splits, p->sm_count, (cudaStream_t)stream,
                  kvp::kLaunchAttention, &P);
    if (rc) return rc;
    rc = dispatch(variant, L.head_dim, G, &p->tmap[layout], &a, num_splits, p->sm_count, (cudaStream_t)stream,
                  kvp::kLaunchCombine, &P);
    if (rc) return rc;
    kvp_note_cascade_combine(stream, KvpCascadeNote{workspace, a.skip, flags, ws + plan_off});
    if (ov.on) p->overlapped.fetch_add(1, std::memory_order_relaxed);
    return KV_OK;
}

}  // namespace

extern "C" {

int paged_decode_attn(kv_pool *p, int layout, const uint16_t *q, uint16_t *out, const int32_t *dev_table,
                      const int32_t *dev_ctx_lens, int max_blocks, int S, int Hq, float scale, int num_splits,
                      void *workspace, size_t ws_bytes, void *stream)
{
    return attn_call(p, layout, q, nullptr, nullptr, out, dev_table, dev_ctx_lens, max_blocks, S, Hq, scale,
                     num_splits, workspace, ws_bytes, stream);
}

int paged_decode_attn_append(kv_pool *p, int layout, const uint16_t *q, const uint16_t *k_new,
                             const uint16_t *v_new, uint16_t *out, const int32_t *dev_table,
                             const int32_t *dev_ctx_lens, int max_blocks, int S, int Hq, float scale,
                             int num_splits, void *workspace, size_t ws_bytes, void *stream)
{
    if (!k_new || !v_new) return KV_ERR_INVALID_ARG;
    return attn_call(p, layout, q, k_new, v_new, out, dev_table, dev_ctx_lens, max_blocks, S, Hq, scale,
                     num_splits, workspace, ws_bytes, stream);
}

int paged_decode_attn_seqtab(kv_pool *p, kv_seqtab *t, const uint16_t *q, const uint16_t *k_new,
                             const uint16_t *v_new, uint16_t *out, int32_t *dev_table, int32_t *dev_ctx_lens, int S,
                             int Hq, float scale, int num_splits, void *workspace, size_t ws_bytes, void *stream)
{
    if (!p || !t || t->pool != p || !dev_table || !dev_ctx_lens || S < 0 || S > t->S) return KV_ERR_INVALID_ARG;
    if ((!k_new) != (!v_new)) return KV_ERR_INVALID_ARG;
    const size_t words = (size_t)t->S + 2 * t->changed.size();
    if (t->full_dirty || words > (size_t)kvp::kSyncWords || S == 0) {
        // too much to carry with the launch (or nothing to launch): the
        // separate sync kernel (or a whole-table copy), then the plain call
        int rc = kv_seqtab_sync(t, dev_table, dev_ctx_lens, stream);
        if (rc) return rc;
        return attn_call(p, t->layout, q, k_new, v_new, out, dev_table, dev_ctx_lens, t->max_blocks, S, Hq, scale,
                         num_splits, workspace, ws_bytes, stream);
    }
    const FusedSync sync{t, dev_table, dev_ctx_lens};
    return attn_call(p, t->layout, q, k_new, v_new, out, dev_table, dev_ctx_lens, t->max_blocks, S, Hq, scale,
                     num_splits, workspace, ws_bytes, stream, nullptr, &sync);
}

// One launch-ready batch of paged_decode_attn_multi.
struct MultiItem {
    kvp::AttnArgs a;
    int variant, D, G, layout, P;
};

// paged_decode_attn(_append) arguments of one batch checked and turned into
// launch parameters; nothing is launched.  S == 0 gives *skip = true.
int prepare_plain(kv_pool *p, const kv_attn_batch &b, MultiItem *it, bool *skip)
{
    int G = 0;
    *skip = false;
    if (!std::isfinite(b.scale)) return KV_ERR_INVALID_ARG;
    int rc = attn_shape(p, b.layout, b.S, b.Hq, b.max_blocks, &G);
    if (rc) return rc;
    if (b.S == 0) {
        *skip = true;
        return KV_OK;
    }
    if (!b.q || !b.out || !b.dev_table || !b.dev_ctx_lens || !aligned16(b.q) || !aligned16(b.out))
        return KV_ERR_INVALID_ARG;
    if ((b.k_new || b.v_new) && (!b.k_new || !b.v_new || !aligned16(b.k_new) || !aligned16(b.v_new)))
        return KV_ERR_INVALID_ARG;
    if (p->sm_count <= 0) return KV_ERR_CUDA;
    const kv_layout &L = p->desc.layouts[b.layout];
    kvp::AttnArgs &a = it->a;
    a = kvp::AttnArgs{};
    a.q = b.q;
    a.out = b.out;
    a.k_new = b.k_new;
    a.v_new = b.v_new;
    a.pool = reinterpret_cast<uint16_t *>(p->desc.device_base);
    a.table = b.dev_table;
    a.ctx_lens = b.dev_ctx_lens;
    a.err = p->desc.device_error;
    a.rows_per_page = (int64_t)(p->page_bytes / (2ull * L.head_dim));
    a.pool_pages = p->n_pages;
    a.pages_per_block = p->pages_per_block[b.layout];
    a.max_blocks = b.max_blocks;
    a.S = b.S;
    a.Hkv = L.num_kv_heads;
    a.bs = p->desc.block_size;
    a.qk_scale = b.scale * 1.4426950408889634f;
    it->variant = pick_variant(p, G);
    it->D = L.head_dim;
    it->G = G;
    it->layout = b.layout;
    int P = 0;
    rc = dispatch(it->variant, L.head_dim, G, nullptr, &a, 0, p->sm_count, nullptr, kvp::kLaunchQuery, &P);
    if (rc) return rc;
    it->P = P;
    size_t part_off;
    const size_t need = ws_layout(b.S, L.num_kv_heads, G, L.head_dim, P, &part_off);
    if (!b.workspace || b.ws_bytes < need || ((uintptr_t)b.workspace & 255u)) return KV_ERR_WORKSPACE;
    a.ws_run = reinterpret_cast<int2 *>(b.workspace);
    a.ws_part = reinterpret_cast<float *>(reinterpret_cast<uint8_t *>(b.workspace) + part_off);
    return ensure_tmap(p, b.layout);
}

int paged_decode_attn_multi(kv_pool *p, int n, const kv_attn_batch *batches, void *stream)
{
    if (!p || n < 0 || (n > 0 && !batches)) return KV_ERR_INVALID_ARG;
    // every batch is checked before anything is launched
    std::vector<MultiItem> items;
    items.reserve((size_t)n);
    for (int i = 0; i < n; ++i) {
        MultiItem it;
        bool skip = false;
        int rc = prepare_plain(p, batches[i], &it, &skip);
        if (rc) return rc;
        if (!skip) items.push_back(it);
    }
    cudaStream_t st = (cudaStream_t)stream;
    int P = 0;
    if (items.size() == 1) {
        MultiItem &it = items[0];
        return dispatch(it.variant, it.D, it.G, &p->tmap[it.layout], &it.a, it.P, p->sm_count, st,
                        kvp::kLaunchBoth, &P);
    }
    // the decode kernels as a chain (each later one starts on the SMs the one
    // before frees and waits for it at its end), then the combines
    for (size_t i = 0; i < items.size(); ++i) {
        MultiItem &it = items[i];
        it.a.chain = i == 0 ? 1 : 2;
        int rc = dispatch(it.variant, it.D, it.G, &p->tmap[it.layout], &it.a, it.P, p->sm_count, st,
                          kvp::kLaunchAttention, &P);
        if (rc) return rc;
    }
    for (MultiItem &it : items) {
        int rc = dispatch(it.variant, it.D, it.G, &p->tmap[it.layout], &it.a, it.P, p->sm_count, st,
                          kvp::kLaunchCombine, &P);
        if (rc) return rc;
    }
    return KV_OK;
}

}  // extern "C"

extern "C" int paged_decode_attn_cascade(kv_pool *p, int layout, const uint16_t *q, const uint16_t *k_new,
                                         const uint16_t *v_new, uint16_t *out, const int32_t *dev_table,
                                         const int32_t *dev_ctx_lens, int max_blocks, int S, int Hq, float scale,
                                         const kv_prefix_group *groups, int n_groups, const int32_t *members,
                                         void *workspace, size_t ws_bytes, void *stream)
{
    if (n_groups < 0 || (!k_new) != (!v_new)) return KV_ERR_INVALID_ARG;
    if (n_groups == 0)
        return attn_call(p, layout, q, k_new, v_new, out, dev_table, dev_ctx_lens, max_blocks, S, Hq, scale, 0,
                         workspace, ws_bytes, stream);
    const CascadePlan plan{groups, n_groups, members};
    return attn_call(p, layout, q, k_new, v_new, out, dev_table, dev_ctx_lens, max_blocks, S, Hq, scale, 0,
                     workspace, ws_bytes, stream, &plan);
}

extern "C" int paged_decode_attn_cascade_seqtab(kv_pool *p, kv_seqtab *t, const uint16_t *q, const uint16_t *k_new,
                                                const uint16_t *v_new, uint16_t *out, int32_t *dev_table,
                                                int32_t *dev_ctx_lens, int S, int Hq, float scale,
                                                const kv_prefix_group *groups, int n_groups, const int32_t *members,
                                                void *workspace, size_t ws_bytes, void *stream)
{
    if (!p || !t || t->pool != p || !dev_table || !dev_ctx_lens || S < 0 || S > t->S) return KV_ERR_INVALID_ARG;
    if (n_groups < 0 || (!k_new) != (!v_new)) return KV_ERR_INVALID_ARG;
    if (n_groups == 0)
        return paged_decode_attn_seqtab(p, t, q, k_new, v_new, out, dev_table, dev_ctx_lens, S, Hq, scale, 0,
                                        workspace, ws_bytes, stream);
    if (S == 0) return kv_seqtab_sync(t, dev_table, dev_ctx_lens, stream);
    const CascadePlan plan{groups, n_groups, members};
    const FusedSync sync{t, dev_table, dev_ctx_lens};
    return attn_call(p, t->layout, q, k_new, v_new, out, dev_table, dev_ctx_lens, t->max_blocks, S, Hq, scale, 0,
                     workspace, ws_bytes, stream, &plan, &sync);
}
