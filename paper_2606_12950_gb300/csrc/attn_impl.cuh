// attn_impl.cuh -- paged decode attention kernel for sm_103a.
//
// One decode query per (sequence, query head) attends over the sequence's
// cached K/V (the decode phase, paper §II "LLM inference cost model"), which
// sits in fixed-size blocks of one shared pool reached through a per-sequence
// block table (§II / §III-C).  Per (s, h), with g = h / G:
//     out = sum_j softmax_j(scale * q . K_j) V_j
// evaluated with an online softmax in base 2 and fp32 accumulation.
//
// Work decomposition (all decided on the device from the lengths):
//   unit  = one 16-token tile of one (sequence, KV head) run; a run of n
//           tokens has ceil(n/16) units; units are ordered (s, g, tile).
//   part  = one of NP = P * 8 equal contiguous unit ranges [i*W/NP,
//           (i+1)*W/NP), one per warp of the P resident CTAs: every warp
//           streams the same number of bytes (+-1 tile) whatever the length
//           distribution.
//   piece = the part of one run inside one part.  A run covered by one part
//           is finished in place; a run cut by part boundaries leaves one
//           fp32 partial (max, sum, unnormalised output) per part, which the
//           combine kernel below merges in part order.
// Inside a CTA each of the 8 warps is one part of that split: it streams its
// own contiguous range of units through its own shared-memory stage, issuing
// its own 2-D TMA loads (128-byte swizzle) of each unit's K and V tiles with
// one mbarrier for K and one for V: the next unit's K streams in while the
// warp does softmax and P.V on the current one, the next V while it does the
// next q.K.  (Measured on GB300: one issuing thread per SM cannot keep HBM
// busy with these 2 KB boxes; one per warp can.)  The pool rows of the CTA's
// units are resolved from the block table in the prologue, while the memory
// system is idle, so no table load sits on the streaming path, and each
// run's q rows (and, for the run's last tile, this step's new K/V rows) are
// staged into the warp's shared buffers by cp.async one piece ahead.  A run
// that ends inside a warp's range is written out by that warp directly; no
// state is merged between warps of a CTA.
//
// Grid-to-grid order: the kernel is launched as a programmatic dependent.
// Alone it releases the next grid and waits for the one before; as part of
// a chain (beside the shared-prefix kernel, or the later batches of several
// co-located ones) it starts without waiting, reads what earlier grids wrote
// through L2 only, and waits at its end (AttnArgs::chain).  Right after a
// split-K combine (step overlap) it starts without waiting too, while the
// combine finishes, and waits before its first write of the output or the
// workspace, which the combine uses.  The step's
// table sync may ride in its parameters (AttnArgs::sync_words); a grid
// alone then computes its work split from those lengths before its wait.
//
// Two compute variants share this skeleton:
//   FmaCompute : CUDA-core FFMA2 dot products and weighted sums.
//   MmaCompute : warp-level tensor-core MMA (m16n8k16 bf16 -> fp32); tokens
//                on M, the query-head group on N (padded to 8), d on K for
//                q.K and on M for P.V; P is moved from accumulator layout to
//                operand layout with movmatrix.
#pragma once

#include <cstdint>

#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include "kvpool.h"
#include "ptx.cuh"

namespace kvp {

// Warps per CTA, each streaming and computing its own units: up to kWarps
// (AttnArgs::nwarps).  Two CTAs of six warps on an SM keep 12 units in
// flight there, which config 2 (64 sequences on all 152 SMs) streams
// fastest; beside the shared-prefix kernel, on fewer SMs, eight do.
constexpr int kWarps = 8;
constexpr int kThreads = kWarps * 32;
constexpr int kPlainWarps = 6;
constexpr int kStages = 1;  // units in flight per warp (each a K and a V tile)
constexpr int kTile = 16;                         // tokens per unit
constexpr int kMinUnitsPerPart = 4;
constexpr uint32_t kHalfBytes = kTile * 128;      // one 64-column box: 16 rows x 128 B
constexpr uint64_t kWaitLimitNs = 2000000000ull;  // bounded mbarrier waits: 2 s

// Loads of data written by earlier grids: through L2 only (ld.global.cg) when
// the kernel did not wait for the grid before it (a chained grid: beside the
// shared-prefix kernel, a later batch of paged_decode_attn_multi, or a step
// overlapping the previous step's combine), so that no line an earlier
// kernel left in this SM's L1 is read; plain otherwise.
template <class T>
__device__ __forceinline__ T ld_prior(const T *p, bool l2_only)
{
    return l2_only ? __ldcg(p) : *p;
}

// Words of a table sync carried by the decode kernel's parameters (lengths,
// then (flat index, value) pairs of changed table entries): 512 bytes, which
// every launch carries.  A 1.8 KB block cost the launch more than the
// separate sync kernel saved (measured on config 2).
constexpr int kSyncWords = 128;

struct AttnArgs {
    const uint16_t *q;
    uint16_t *out;
    const uint16_t *k_new;   // fused append: this step's K/V rows [S][Hkv][d], or null
    const uint16_t *v_new;
    uint16_t *pool;          // pool base (rows of d bf16), for the fused append's writes
    const int32_t *table;
    const int32_t *ctx_lens;
    int32_t *err;
    float *ws_part;
    int2 *ws_run;            // per run: (first part, parts) if split, else (part, 0)
    int64_t rows_per_page;   // page_bytes / (d * 2)
    int64_t pool_pages;
    int32_t pages_per_block;
    int32_t max_blocks;
    int32_t S;
    int32_t Hkv;
    int32_t bs;
    int32_t rows_cap;        // units whose pool rows are resolved up front
    int32_t P;               // CTAs
    int32_t nwarps;          // warps per CTA (<= kWarps), one part each
    float qk_scale;          // scale * log2(e)
    // shared-prefix (cascade) mode: tokens of each sequence's prefix handled
    // by the prefix kernel ([S], multiples of 16; null = none), its records
    // and key-split count (read by the combine)
    const int32_t *skip;
    const float *ws_pre;
    int32_t KS;
    // place in a chain of grids: 0 alone (release the next grid, then wait
    // for the one before); 1 first of a chain (wait, then release: the next
    // grid relies on this wait); 2 chained (release, no wait at the start,
    // a wait at every exit: see the kernel); 3 right after a split-K combine
    // of this library, which released this grid only after its own wait, so
    // every grid before that combine has completed (release, no wait at the
    // start, a wait before the first write of the output or the workspace,
    // which the combine still uses, and at every exit); 4 beside the
    // shared-prefix kernel while the previous step's shared-prefix combine
    // finishes (release, no wait at the start; the plan kernel's two flags,
    // below, stand in for the waits: the first before anything the plan
    // kernel writes is read, the second before the first write of the output
    // or the workspace; a wait for the prefix grid at every exit)
    int32_t chain;
    // chain 4: the plan kernel sets flags[0] = epoch once the plan, the
    // skips and the table sync are written, and flags[1] = epoch once every
    // grid before it has completed
    const uint64_t *flags;
    uint64_t epoch;
    // fused table sync (paged_decode_attn_seqtab): this step's lengths of
    // rows [0, sync_nlens) and its changed table entries travel here.  The
    // kernel takes the lengths and those entries from here, and the CTAs
    // write them to sync_lens / sync_table for later kernels.  Null: none.
    int32_t *sync_table;
    int32_t *sync_lens;
    int32_t sync_nlens;
    int32_t sync_npatch;
    int32_t sync_words[kSyncWords];
};

__device__ __forceinline__ void report(int32_t *err, int code) { atomicCAS(err, 0, code); }

// bounded wait on an mbarrier phase; a wait that exceeds the limit records
// KV_ERR_DEVICE_TIMEOUT and makes every later wait of this warp return at once
__device__ __forceinline__ void wait_phase(uint32_t bar, uint32_t parity, int32_t *err, bool &dead)
{
    if (dead) return;
    if (mbar_try_wait(bar, parity)) return;
    uint64_t t0 = global_timer_ns();
    for (uint32_t it = 1;; ++it) {
        if (mbar_try_wait(bar, parity)) return;
        if ((it & 1023u) == 0 && global_timer_ns() - t0 > kWaitLimitNs) {
            report(err, KV_ERR_DEVICE_TIMEOUT);
            dead = true;
            return;
        }
    }
}

// bounded wait until another grid has stored `epoch` in *flag (release
// store; this load acquires); a wait past the limit records
// KV_ERR_DEVICE_TIMEOUT and returns
__device__ __forceinline__ void wait_flag(const uint64_t *flag, uint64_t epoch, int32_t *err)
{
    if (ld_acquire_gpu(flag) == epoch) return;
    const uint64_t t0 = global_timer_ns();
    for (uint32_t it = 1;; ++it) {
        __nanosleep(64);
        if (ld_acquire_gpu(flag) == epoch) return;
        if ((it & 255u) == 0 && global_timer_ns() - t0 > kWaitLimitNs) {
            report(err, KV_ERR_DEVICE_TIMEOUT);
            return;
        }
    }
}

// shared-memory byte offset of 16-byte chunk c (8 bf16 of columns 8c..8c+7)
// of tile row r, in the 128-byte-swizzled layout TMA writes
__device__ __forceinline__ uint32_t swz(int r, int c)
{
    return (uint32_t)((c >> 3) * kHalfBytes + r * 128 + (((c & 7) ^ (r & 7)) << 4));
}

__device__ __forceinline__ float bf_lo(uint32_t w) { return __uint_as_float(w << 16); }
__device__ __forceinline__ float bf_hi(uint32_t w) { return __uint_as_float(w & 0xFFFF0000u); }

// ------------------------------------------------------------ CUDA cores ---
template <int D, int G>
struct FmaCompute {
    static constexpr int kMinBlocks = 1;                     // registers allow one CTA per SM
    static constexpr int LPT = (G * D / 8 <= 64) ? 8 : 16;  // lanes per token
    static constexpr int EPL = D / LPT;                      // elements per lane
    static constexpr int NCH = EPL / 8;                      // 16-byte chunks per lane
    static constexpr int NGRP = 32 / LPT;                    // tokens in flight per warp
    static constexpr int TPG = kTile / NGRP;                 // tokens per group per tile
    static_assert(EPL % 8 == 0, "lane slice must be whole 16-byte chunks");

    float2 q[G][EPL / 2];
    float2 o[G][EPL / 2];
    float m[G];
    float l[G];
    float p[TPG][G];
    int grp, sub, nv;

    // qrow: the run's G query rows, staged in shared memory
    __device__ __forceinline__ void begin(const uint16_t *qrow, float qk_scale, int lane)
    {
        grp = lane / LPT;
        sub = lane % LPT;
#pragma unroll
        for (int h = 0; h < G; ++h) {
#pragma unroll
            for (int j = 0; j < NCH; ++j) {
                const int c = sub + j * LPT;
                uint4 w = *reinterpret_cast<const uint4 *>(qrow + h * D + c * 8);
                uint32_t ws[4] = {w.x, w.y, w.z, w.w};
#pragma unroll
                for (int e = 0; e < 4; ++e)
                    q[h][j * 4 + e] = make_float2(bf_lo(ws[e]) * qk_scale, bf_hi(ws[e]) * qk_scale);
            }
#pragma unroll
            for (int e = 0; e < EPL / 2; ++e) o[h][e] = make_float2(0.f, 0.f);
            m[h] = -INFINITY;
            l[h] = 0.f;
        }
    }

    // q.K for the tile's tokens, online-softmax update, weights p
    __device__ __forceinline__ void qk(const uint8_t *Ks, int nvalid)
    {
        nv = nvalid;
        float sc[TPG][G];
#pragma unroll
        for (int i = 0; i < TPG; ++i) {
            const int t = grp + i * NGRP;
            float2 acc[G];
#pragma unroll
            for (int h = 0; h < G; ++h) acc[h] = make_float2(0.f, 0.f);
#pragma unroll
            for (int j = 0; j < NCH; ++j) {
                uint4 w = *reinterpret_cast<const uint4 *>(Ks + swz(t, sub + j * LPT));
                uint32_t ws[4] = {w.x, w.y, w.z, w.w};
#pragma unroll
                for (int e = 0; e < 4; ++e) {
                    float2 kv = make_float2(bf_lo(ws[e]), bf_hi(ws[e]));
#pragma unroll
                    for (int h = 0; h < G; ++h) acc[h] = __ffma2_rn(q[h][j * 4 + e], kv, acc[h]);
                }
            }
#pragma unroll
            for (int h = 0; h < G; ++h) sc[i][h] = acc[h].x + acc[h].y;
        }
        // dot products are split over LPT lanes: butterfly sum
#pragma unroll
        for (int off = 1; off < LPT; off <<= 1)
#pragma unroll
            for (int i = 0; i < TPG; ++i)
#pragma unroll
                for (int h = 0; h < G; ++h) sc[i][h] += __shfl_xor_sync(0xffffffffu, sc[i][h], off);
        float tmax[G];
#pragma unroll
        for (int h = 0; h < G; ++h) tmax[h] = -INFINITY;
#pragma unroll
        for (int i = 0; i < TPG; ++i) {
            const bool ok = grp + i * NGRP < nvalid;
#pragma unroll
            for (int h = 0; h < G; ++h) {
                sc[i][h] = ok ? sc[i][h] : -INFINITY;
                tmax[h] = fmaxf(tmax[h], sc[i][h]);
            }
        }
#pragma unroll
        for (int off = LPT; off < 32; off <<= 1)
#pragma unroll
            for (int h = 0; h < G; ++h) tmax[h] = fmaxf(tmax[h], __shfl_xor_sync(0xffffffffu, tmax[h], off));
        // lazy rescale: keep the running max unless the tile exceeds it by
        // more than 2^8 (o and l share the stale max, so the ratio is exact)
#pragma unroll
        for (int h = 0; h < G; ++h) {
            if (tmax[h] > m[h] + 8.f) {
                const float a = fast_exp2(m[h] - tmax[h]);
                l[h] *= a;
#pragma unroll
                for (int e = 0; e < EPL / 2; ++e) o[h][e] = make_float2(o[h][e].x * a, o[h][e].y * a);
                m[h] = tmax[h];
            }
        }
#pragma unroll
        for (int i = 0; i < TPG; ++i)
#pragma unroll
            for (int h = 0; h < G; ++h) {
                p[i][h] = fast_exp2(sc[i][h] - m[h]);
                l[h] += p[i][h];
            }
    }

    // o += p * V for the tile's valid tokens
    __device__ __forceinline__ void pv(uint8_t *Vs)
    {
#pragma unroll
        for (int i = 0; i < TPG; ++i) {
            const int t = grp + i * NGRP;
            if (t < nv) {
#pragma unroll
                for (int j = 0; j < NCH; ++j) {
                    uint4 w = *reinterpret_cast<const uint4 *>(Vs + swz(t, sub + j * LPT));
                    uint32_t ws[4] = {w.x, w.y, w.z, w.w};
#pragma unroll
                    for (int e = 0; e < 4; ++e) {
                        float2 vv = make_float2(bf_lo(ws[e]), bf_hi(ws[e]));
#pragma unroll
                        for (int h = 0; h < G; ++h)
                            o[h][j * 4 + e] = __ffma2_rn(make_float2(p[i][h], p[i][h]), vv, o[h][j * 4 + e]);
                    }
                }
            }
        }
    }

    // end of a piece: the bf16 output o / l (whole run in this warp), or the
    // fp32 partial (o unnormalised, m, l) of this warp's part of the run
    __device__ __forceinline__ void store(uint16_t *orow, float *slot, bool split, int lane)
    {
#pragma unroll
        for (int off = LPT; off < 32; off <<= 1)
#pragma unroll
            for (int h = 0; h < G; ++h) {
                l[h] += __shfl_xor_sync(0xffffffffu, l[h], off);
#pragma unroll
                for (int e = 0; e < EPL / 2; ++e) {
                    o[h][e].x += __shfl_xor_sync(0xffffffffu, o[h][e].x, off);
                    o[h][e].y += __shfl_xor_sync(0xffffffffu, o[h][e].y, off);
                }
            }
        if (grp == 0) {
#pragma unroll
            for (int h = 0; h < G; ++h)
#pragma unroll
                for (int j = 0; j < NCH; ++j) {
                    const int c = sub + j * LPT;
                    if (!split) {
                        uint32_t w[4];
#pragma unroll
                        for (int e = 0; e < 4; ++e) {
                            __nv_bfloat162 b2 =
                                __floats2bfloat162_rn(o[h][j * 4 + e].x / l[h], o[h][j * 4 + e].y / l[h]);
                            w[e] = *reinterpret_cast<uint32_t *>(&b2);
                        }
                        *reinterpret_cast<uint4 *>(orow + h * D + c * 8) = make_uint4(w[0], w[1], w[2], w[3]);
                    } else {
                        float4 *dst = reinterpret_cast<float4 *>(slot + h * D + c * 8);
                        dst[0] = make_float4(o[h][j * 4 + 0].x, o[h][j * 4 + 0].y, o[h][j * 4 + 1].x, o[h][j * 4 + 1].y);
                        dst[1] = make_float4(o[h][j * 4 + 2].x, o[h][j * 4 + 2].y, o[h][j * 4 + 3].x, o[h][j * 4 + 3].y);
                    }
                }
        }
        if (split && lane == 0) {
#pragma unroll
            for (int h = 0; h < G; ++h) {
                slot[G * D + h] = m[h];
                slot[G * D + G + h] = l[h];
            }
        }
    }
};

// ----------------------------------------------------------- tensor cores --
template <int D, int G>
struct MmaCompute {
    static_assert(G <= 8, "query-head group must fit the n=8 MMA tile");
    static constexpr int kMinBlocks = 2;
    static constexpr int KS = D / 16;
    uint32_t qf[KS][2];  // B operand of q.K: Q^T fragments (bf16x2)
    float acc[KS][4];    // O^T accumulators, 16 d-rows per block
    float m[2], l[2];    // heads 2*tig, 2*tig+1
    uint32_t pb0, pb1;   // B operand of P.V (P^T fragments)
    float qk_scale;
    int gid, tig, lane_, nv;

    // qrow: the run's G query rows, staged in shared memory
    __device__ __forceinline__ void begin(const uint16_t *qrow, float scale, int lane)
    {
        lane_ = lane;
        gid = lane >> 2;
        tig = lane & 3;
        qk_scale = scale;
#pragma unroll
        for (int kk = 0; kk < KS; ++kk) {
            if (gid < G) {
                qf[kk][0] = *reinterpret_cast<const uint32_t *>(qrow + gid * D + kk * 16 + tig * 2);
                qf[kk][1] = *reinterpret_cast<const uint32_t *>(qrow + gid * D + kk * 16 + tig * 2 + 8);
            } else {
                qf[kk][0] = 0u;
                qf[kk][1] = 0u;
            }
#pragma unroll
            for (int e = 0; e < 4; ++e) acc[kk][e] = 0.f;
        }
        m[0] = m[1] = -INFINITY;
        l[0] = l[1] = 0.f;
    }

    __device__ __forceinline__ void qk(const uint8_t *Ks, int nvalid)
    {
        nv = nvalid;
        const uint32_t kbase = smem_u32(Ks);
        const int mat = lane_ >> 3, r8 = lane_ & 7;
        float s[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
        for (int kk = 0; kk < KS; ++kk) {
            uint32_t a0, a1, a2, a3;
            ldmatrix_x4(kbase + swz(r8 + (mat & 1) * 8, kk * 2 + (mat >> 1)), a0, a1, a2, a3);
            mma_bf16_16816(s, a0, a1, a2, a3, qf[kk][0], qf[kk][1]);
        }
        // s[0], s[1]: token gid, heads 2tig, 2tig+1; s[2], s[3]: token gid+8
        const bool ok0 = gid < nvalid, ok1 = gid + 8 < nvalid;
        const float x0 = ok0 ? s[0] * qk_scale : -INFINITY;
        const float x1 = ok0 ? s[1] * qk_scale : -INFINITY;
        const float x2 = ok1 ? s[2] * qk_scale : -INFINITY;
        const float x3 = ok1 ? s[3] * qk_scale : -INFINITY;
        float t0 = fmaxf(x0, x2), t1 = fmaxf(x1, x3);
#pragma unroll
        for (int off = 4; off < 32; off <<= 1) {
            t0 = fmaxf(t0, __shfl_xor_sync(0xffffffffu, t0, off));
            t1 = fmaxf(t1, __shfl_xor_sync(0xffffffffu, t1, off));
        }
        // lazy rescale (see FmaCompute::qk)
        if (t0 > m[0] + 8.f) {
            const float a = fast_exp2(m[0] - t0);
            l[0] *= a;
#pragma unroll
            for (int mb = 0; mb < KS; ++mb) {
                acc[mb][0] *= a;
                acc[mb][2] *= a;
            }
            m[0] = t0;
        }
        if (t1 > m[1] + 8.f) {
            const float a = fast_exp2(m[1] - t1);
            l[1] *= a;
#pragma unroll
            for (int mb = 0; mb < KS; ++mb) {
                acc[mb][1] *= a;
                acc[mb][3] *= a;
            }
            m[1] = t1;
        }
        const float p0 = fast_exp2(x0 - m[0]), p1 = fast_exp2(x1 - m[1]);
        const float p2 = fast_exp2(x2 - m[0]), p3 = fast_exp2(x3 - m[1]);
        l[0] += p0 + p2;
        l[1] += p1 + p3;
        __nv_bfloat162 lo = __floats2bfloat162_rn(p0, p1);
        __nv_bfloat162 hi = __floats2bfloat162_rn(p2, p3);
        pb0 = movmatrix_trans(*reinterpret_cast<uint32_t *>(&lo));
        pb1 = movmatrix_trans(*reinterpret_cast<uint32_t *>(&hi));
    }

    __device__ __forceinline__ void pv(uint8_t *Vs)
    {
        // rows past the context may hold anything (even NaN bit patterns);
        // P is zero there, but 0 * NaN is NaN inside the MMA, so clear them
        if (nv < kTile) {
            const int nchunk = (kTile - nv) * (D / 8);
            for (int idx = lane_; idx < nchunk; idx += 32) {
                const int r = nv + idx / (D / 8);
                const int c = idx % (D / 8);
                *reinterpret_cast<uint4 *>(Vs + swz(r, c)) = make_uint4(0u, 0u, 0u, 0u);
            }
            __syncwarp();
        }
        const uint32_t vbase = smem_u32(Vs);
        const int mat = lane_ >> 3, r8 = lane_ & 7;
#pragma unroll
        for (int mb = 0; mb < KS; ++mb) {
            uint32_t a0, a1, a2, a3;
            ldmatrix_x4_trans(vbase + swz(r8 + (mat >> 1) * 8, mb * 2 + (mat & 1)), a0, a1, a2, a3);
            mma_bf16_16816(acc[mb], a0, a1, a2, a3, pb0, pb1);
        }
    }

    // end of a piece (see FmaCompute::store)
    __device__ __forceinline__ void store(uint16_t *orow, float *slot, bool split, int lane)
    {
#pragma unroll
        for (int off = 4; off < 32; off <<= 1) {
            l[0] += __shfl_xor_sync(0xffffffffu, l[0], off);
            l[1] += __shfl_xor_sync(0xffffffffu, l[1], off);
        }
        const int h0 = 2 * tig, h1 = 2 * tig + 1;
        if (!split) {
#pragma unroll
            for (int mb = 0; mb < KS; ++mb) {
                const int d0 = mb * 16 + gid;
                if (h0 < G) {
                    orow[h0 * D + d0] = __bfloat16_as_ushort(__float2bfloat16_rn(acc[mb][0] / l[0]));
                    orow[h0 * D + d0 + 8] = __bfloat16_as_ushort(__float2bfloat16_rn(acc[mb][2] / l[0]));
                }
                if (h1 < G) {
                    orow[h1 * D + d0] = __bfloat16_as_ushort(__float2bfloat16_rn(acc[mb][1] / l[1]));
                    orow[h1 * D + d0 + 8] = __bfloat16_as_ushort(__float2bfloat16_rn(acc[mb][3] / l[1]));
                }
            }
        } else {
#pragma unroll
            for (int mb = 0; mb < KS; ++mb) {
                const int d0 = mb * 16 + gid;
                if (h0 < G) {
                    slot[h0 * D + d0] = acc[mb][0];
                    slot[h0 * D + d0 + 8] = acc[mb][2];
                }
                if (h1 < G) {
                    slot[h1 * D + d0] = acc[mb][1];
                    slot[h1 * D + d0 + 8] = acc[mb][3];
                }
            }
            if (gid == 0) {
                if (h0 < G) {
                    slot[G * D + h0] = m[0];
                    slot[G * D + G + h0] = l[0];
                }
                if (h1 < G) {
                    slot[G * D + h1] = m[1];
                    slot[G * D + G + h1] = l[1];
                }
            }
        }
        (void)lane;
    }
};

// ----------------------------------------------------------- work units ---
struct Piece {
    int32_t pb, pe;        // piece unit range
    int32_t run_begin;     // unit id of tile 0 of this (s, g) run
    int32_t run_end;
    int32_t s, g, n;       // sequence, KV head, context length
    int32_t skip;          // leading tokens handled by the prefix kernel
};

// Context length of sequence s, read once per CTA in the prologue and clamped
// to the table's reach with the error reported.
__device__ __forceinline__ int32_t load_len(const AttnArgs &a, int s, int32_t *raw_out)
{
    const int32_t raw = a.sync_table ? a.sync_words[s] : ld_prior(a.ctx_lens + s, a.chain >= 2);
    const int32_t cap = a.max_blocks * a.bs;
    *raw_out = raw;
    if (raw < 0 || raw > cap) {
        report(a.err, KV_ERR_DEVICE_BOUNDS);
        return raw < 0 ? 0 : cap;
    }
    return raw;
}

// leading tokens of sequence s (context n) left to the prefix kernel: 0
// outside shared-prefix mode; a value that is not a multiple of 16 in
// [0, n] is reported and clamped
__device__ __forceinline__ int32_t load_skip(const AttnArgs &a, int s, int32_t n)
{
    if (!a.skip) return 0;
    int32_t k = __ldcg(a.skip + s);
    if (k < 0 || k > n || (k % kTile)) {
        report(a.err, KV_ERR_DEVICE_BOUNDS);
        k = k < 0 ? 0 : (k > n ? n : k);
        k -= k % kTile;
    }
    return k;
}

// The CTA's copy of the per-sequence values, after T[0 .. S]: NL[s] = the
// clamped length, with bit 31 set when the stored length was out of range;
// SK[s] = the clamped skip.
__device__ __forceinline__ int32_t seq_len(const int32_t *T, int S, int s) { return T[S + 1 + s] & 0x7fffffff; }
__device__ __forceinline__ bool seq_len_clamped(const int32_t *T, int S, int s) { return T[S + 1 + s] < 0; }
__device__ __forceinline__ int32_t seq_skip(const int32_t *T, int S, int s) { return T[2 * S + 1 + s]; }

// largest s with T[s] <= u; T[s] = first unit of sequence s, T[S] = total,
// so empty sequences (T[s] == T[s+1]) are skipped
__device__ __forceinline__ int find_seq(const int32_t *T, int S, int32_t u)
{
    int lo = 0, hi = S;
    while (hi - lo > 1) {
        const int mid = (lo + hi) >> 1;
        if (T[mid] <= u) lo = mid; else hi = mid;
    }
    return lo;
}

__device__ __forceinline__ void decode_piece(const AttnArgs &a, const int32_t *T, int32_t u, int32_t u1, Piece &p)
{
    const int s = find_seq(T, a.S, u);
    const int32_t nt = (T[s + 1] - T[s]) / a.Hkv;
    const int32_t g = (u - T[s]) / nt;
    p.s = s;
    p.g = g;
    p.n = seq_len(T, a.S, s);
    p.skip = seq_skip(T, a.S, s);
    p.run_begin = T[s] + g * nt;
    p.run_end = p.run_begin + nt;
    p.pb = u;
    p.pe = p.run_end < u1 ? p.run_end : u1;
}

// Block table entry idx (flat): this step's value when the table sync is
// fused into the launch and changed that entry, else the table's.
__device__ __forceinline__ int32_t table_entry(const AttnArgs &a, int64_t idx)
{
    if (a.sync_table) {
        const int32_t *pw = a.sync_words + a.sync_nlens;
        for (int j = 0; j < a.sync_npatch; ++j)
            if (pw[2 * j] == idx) return pw[2 * j + 1];
    }
    return ld_prior(a.table + idx, a.chain >= 2);
}

// Pool row of unit u's K tile (TMA y coordinate; V is Hkv*bs rows further),
// or -1 if the block table names a block outside the pool.
__device__ __forceinline__ int32_t unit_row(const AttnArgs &a, const int32_t *T, int32_t u)
{
    const int s = find_seq(T, a.S, u);
    const int32_t nt = (T[s + 1] - T[s]) / a.Hkv;
    const int32_t within = u - T[s];
    const int32_t g = within / nt;
    const int32_t tok0 = seq_skip(T, a.S, s) + (within - g * nt) * kTile;
    const int32_t phys = table_entry(a, (int64_t)s * a.max_blocks + tok0 / a.bs);
    if (phys < 0 || (int64_t)phys + a.pages_per_block > a.pool_pages) return -1;
    return (int32_t)((int64_t)phys * a.rows_per_page + (tok0 % a.bs) + (int64_t)g * a.bs);
}

// the part (of NP) whose range contains unit u
__device__ __forceinline__ int32_t cta_of(int64_t u, int64_t W, int64_t P)
{
    return (int32_t)(((u + 1) * P - 1) / W);
}

// per-part partial: o[G][D], m[G], l[G], padded to a multiple of 4 floats so
// every record starts 16-byte aligned
template <int D, int G>
__host__ __device__ constexpr uint32_t merge_floats() { return (G * D + 2 * G + 3) / 4 * 4; }

// Load K (which = 0) or V (which = 1) of unit u into this warp's stage;
// completes on `bar`.  Lane 0 only.
template <int D>
__device__ __forceinline__ void issue_half(const CUtensorMap *tmap, const AttnArgs &a, const int32_t *T,
                                           const int32_t *rows, int32_t cu0, int32_t u, int which, uint32_t dst,
                                           uint32_t bar, uint64_t policy)
{
    constexpr int HALVES = D / 64;
    const int32_t k = u - cu0;
    int32_t y = k < a.rows_cap ? rows[k] : unit_row(a, T, u);
    if (y < 0) {
        report(a.err, KV_ERR_DEVICE_BOUNDS);
        mbar_arrive(bar);  // complete the phase without data
        return;
    }
    y += which * a.Hkv * a.bs;
    mbar_arrive_expect_tx(bar, HALVES * kHalfBytes);
#pragma unroll
    for (int h = 0; h < HALVES; ++h) tma_load_2d(dst + h * kHalfBytes, tmap, h * 64, y, bar, policy);
}

template <int D, int G, class Comp>
__global__ void __launch_bounds__(kThreads, Comp::kMinBlocks)
paged_attn_kernel(const __grid_constant__ CUtensorMap tmap, const __grid_constant__ AttnArgs a)
{
    constexpr int HALVES = D / 64;
    constexpr uint32_t TILE_BYTES = HALVES * kHalfBytes;
    constexpr uint32_t STAGE_BYTES = 2 * TILE_BYTES;
    constexpr uint32_t MF = merge_floats<D, G>();
    extern __shared__ uint8_t smem_raw[];
    // stages need 1024-byte alignment for the 128-byte swizzle pattern
    uint8_t *smem = smem_raw + ((1024u - (smem_u32(smem_raw) & 1023u)) & 1023u);
    constexpr uint32_t QB = G * D * 2, AB = 2 * D * 2;  // q rows of a run; its new K and V rows
    const int NW = a.nwarps, NT = NW * 32;  // warps (parts) of this CTA
    uint8_t *stages = smem;                                                              // [NW][kStages][STAGE]
    uint8_t *qbufs = stages + (size_t)NW * kStages * STAGE_BYTES;                        // [NW][QB]
    uint8_t *abufs = qbufs + (size_t)NW * QB;                                            // [NW][AB]
    uint64_t *bars = reinterpret_cast<uint64_t *>(abufs + (size_t)NW * AB);              // K[w][st], V[w][st]
    int32_t *misc = reinterpret_cast<int32_t *>(bars + 2 * NW * kStages);               // [16] scratch
    int32_t *T = misc + 16;                                                              // [S + 1]
    int32_t *NL = T + a.S + 1;                                                           // [S]
    int32_t *SK = NL + a.S;                                                              // [S]
    int32_t *rows = SK + a.S;                                                            // [rows_cap]

    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int S = a.S, Hkv = a.Hkv, Hq = a.Hkv * G;

    if (tid == 0) {
        for (int i = 0; i < 2 * NW * kStages; ++i) mbar_init(smem_u32(&bars[i]), 1);
        fence_mbar_init();
    }
    if (tid == 32) prefetch_tensormap(&tmap);
    // Launched as a programmatic dependent: everything above touches only
    // this CTA.  Alone (chain 0), release the next grid and wait here for
    // the grid before (lengths, table, pool writes).  A chained grid (chain
    // 2: the decode kernel beside the shared-prefix kernel, or the second
    // and later batches of paged_decode_attn_multi) follows a grid that
    // released it only after its own wait had seen every earlier grid
    // complete; it does not wait for that grid here, so the two run side by
    // side (the later one's CTAs take the SMs the earlier one frees), and
    // waits for it at every exit (`chained`), so that a combine after it
    // sees every chained grid's records.  Data from earlier grids is then
    // read through L2 (ld_prior).  The first grid of a chain (chain 1)
    // waits before it releases the next.  With the lengths carried in the
    // parameters (fused table sync) and no shared prefix, the first prologue
    // below reads nothing that another grid writes and writes only shared
    // memory, so a grid alone runs it before its wait, beside the grid
    // before it (`early`).  After a combine (chain 3) nothing before that
    // combine is still running: the kernel reads and writes the table, the
    // lengths and the pool at once, and each thread waits for the combine
    // (`ready`) before it first writes the output or the workspace.  Beside
    // the prefix kernel of a step that overlaps the previous step's
    // shared-prefix combine (chain 4), the plan kernel's flags take the place
    // of those waits: the first before the lengths, skips and table are read,
    // the second before the first write of the output or the workspace.
    const bool early = a.sync_table != nullptr && a.skip == nullptr && (a.chain == 0 || a.chain == 3);
    if (a.chain != 1) grid_launch_dependents();
    if (a.chain <= 1 && !early) grid_dependency_wait();
    if (a.chain == 1) grid_launch_dependents();
    const bool chained = a.chain >= 2;
    bool ready = a.chain != 3 && a.chain != 4;  // the output and the workspace may be written
    auto make_ready = [&]() {
        if (!ready) {
            if (a.chain == 4)
                wait_flag(a.flags + 1, a.epoch, a.err);
            else
                grid_dependency_wait();
            ready = true;
        }
    };
    if (a.chain == 4) {
        if (tid == 0) wait_flag(a.flags, a.epoch, a.err);
        __syncthreads();
    }
    auto write_sync = [&]() {
        // fused table sync: the grids before have completed (the wait
        // before this), and no CTA of this grid reads what is written here
        const int stride = a.P * NT, i0 = (int)blockIdx.x * NT + tid;
        for (int i = i0; i < a.sync_nlens; i += stride) a.sync_lens[i] = a.sync_words[i];
        const int32_t *pw = a.sync_words + a.sync_nlens;
        for (int j = i0; j < a.sync_npatch; j += stride) a.sync_table[pw[2 * j]] = pw[2 * j + 1];
    };
    if (a.sync_table && !early) write_sync();

    // ---- prologue 1: T[s] = first unit of sequence s ----
    {
        const int per = (S + NT - 1) / NT;
        const int lo = min(S, tid * per), hi = min(S, lo + per);
        int32_t local = 0;
        for (int s = lo; s < hi; ++s) {
            int32_t raw;
            const int32_t n = load_len(a, s, &raw);
            const int32_t k = load_skip(a, s, n);
            NL[s] = n | (raw != n ? (int32_t)0x80000000 : 0);
            SK[s] = k;
            const int32_t ne = n - k;
            local += ((ne + kTile - 1) / kTile) * Hkv;
        }
        int32_t incl = local;
#pragma unroll
        for (int off = 1; off < 32; off <<= 1) {
            const int32_t v = __shfl_up_sync(0xffffffffu, incl, off);
            if (lane >= off) incl += v;
        }
        if (lane == 31) misc[warp] = incl;
        __syncthreads();
        int32_t base = 0;
        for (int w = 0; w < warp; ++w) base += misc[w];
        int32_t run = base + incl - local;
        for (int s = lo; s < hi; ++s) {  // this thread's own NL / SK entries
            T[s] = run;
            run += ((seq_len(T, S, s) - seq_skip(T, S, s) + kTile - 1) / kTile) * Hkv;
        }
        if (tid == 0) {
            int32_t tot = 0;
            for (int w = 0; w < NW; ++w) tot += misc[w];
            T[S] = tot;
        }
        if (early) {
            if (a.chain == 0) grid_dependency_wait();
            write_sync();
        }
        for (int s = lo; s < hi; ++s) {  // sequences with no tile: writes after any wait
            const int32_t n = NL[s] & 0x7fffffff, ne = n - SK[s];
            if (ne != 0 || (s % a.P) != (int)blockIdx.x) continue;
            make_ready();
            // the fused append needs the new token outside a shared prefix
            if (a.skip && a.k_new && n > 0) report(a.err, KV_ERR_DEVICE_BOUNDS);
            // an empty context has no softmax: its output is defined as
            // zero; a sequence whose whole context is a shared prefix gets
            // its output from the prefix records alone
            if (n == 0)
                for (int i = 0; i < Hq * D; ++i) a.out[(int64_t)s * Hq * D + i] = 0;
            for (int g = 0; g < Hkv; ++g) a.ws_run[(int64_t)s * Hkv + g] = make_int2(0, 0);
        }
        __syncthreads();
    }

    // The W units are cut into NP = min(P * NW, W) equal parts; part i is
    // [i*W/NP, (i+1)*W/NP) and belongs to warp i % NW of CTA i / NW.
    // With NP <= W every part is non-empty, so a run's contributors are
    // exactly the parts part_of(first unit) .. part_of(last unit).  A part
    // gets at least kMinUnitsPerPart units when the batch is small (fewer
    // partials to write and merge; enough warps still stream to fill HBM).
    const int64_t W = T[S];
    const int64_t np_min = W > 0 ? (W / kMinUnitsPerPart > 0 ? W / kMinUnitsPerPart : 1) : 0;
    const int64_t NP = np_min < (int64_t)a.P * NW ? np_min : (int64_t)a.P * NW;
    const int64_t first_part = (int64_t)blockIdx.x * NW;
    if (first_part >= NP) {
        if (chained) grid_dependency_wait();
        return;
    }
    const int64_t last_part = first_part + NW < NP ? first_part + NW : NP;  // exclusive
    const int32_t cu0 = (int32_t)(first_part * W / NP);                             // this CTA's units
    const int32_t cu1 = (int32_t)(last_part * W / NP);

    // ---- prologue 2: resolve the block table for this CTA's units while the
    // memory system is idle (later lookups would queue behind the TMA stream)
    {
        const int32_t nr = min(cu1 - cu0, a.rows_cap);
        for (int32_t k = tid; k < nr; k += NT) rows[k] = unit_row(a, T, cu0 + k);
        __syncthreads();
    }

    const int64_t part = first_part + warp;
    if (part >= NP) {  // no CTA-wide barrier below this point
        if (chained) grid_dependency_wait();
        return;
    }
    const int32_t u0 = (int32_t)(part * W / NP);
    const int32_t u1 = (int32_t)((part + 1) * W / NP);

    const uint64_t policy = l2_policy_evict_first();
    // stage st of this warp: its K and V tiles and their barriers
    uint8_t *wstage = stages + (size_t)warp * kStages * STAGE_BYTES;
    auto k_of = [&](int st) { return wstage + (size_t)st * STAGE_BYTES; };
    auto bk_of = [&](int st) { return smem_u32(&bars[warp * kStages + st]); };
    auto bv_of = [&](int st) { return smem_u32(&bars[(NW + warp) * kStages + st]); };

    if (lane == 0) {
        for (int st = 0; st < kStages && u0 + st < u1; ++st) {
            issue_half<D>(&tmap, a, T, rows, cu0, u0 + st, 0, smem_u32(k_of(st)), bk_of(st), policy);
            issue_half<D>(&tmap, a, T, rows, cu0, u0 + st, 1, smem_u32(k_of(st) + TILE_BYTES), bv_of(st), policy);
        }
    }
    // A run's q rows and, for the run's last tile, its new K/V rows are staged
    // in this warp's shared buffers by cp.async one piece ahead, so that no
    // piece start or append waits on a dependent global load.
    uint8_t *qb = qbufs + (size_t)warp * QB;
    uint8_t *ab = abufs + (size_t)warp * AB;
    const uint32_t qb_addr = smem_u32(qb), ab_addr = smem_u32(ab);
    {
        const int s0 = find_seq(T, S, u0);
        const int32_t nt0 = (T[s0 + 1] - T[s0]) / Hkv;
        const uint16_t *src = a.q + ((int64_t)s0 * Hq + (int64_t)((u0 - T[s0]) / nt0) * G) * D;
        for (uint32_t c = lane; c < QB / 16; c += 32) cp_async16(qb_addr + c * 16, src + c * 8);
        cp_async_commit();
    }

    bool dead = false;
    uint32_t consumed = 0;
    int32_t u = u0;
    while (u < u1) {
        Piece pc;
        decode_piece(a, T, u, u1, pc);
        cp_async_wait_all();  // this piece's q rows
        __syncwarp();
        Comp comp;
        comp.begin(reinterpret_cast<const uint16_t *>(qb), a.qk_scale, lane);
        __syncwarp();  // every lane holds its q fragments: the buffer may be refilled
        // fused append: the run's last tile holds position n-1, whose K/V row
        // is this step's new token; this warp alone reads that tile
        const bool app_run = a.k_new != nullptr && pc.pe == pc.run_end && !seq_len_clamped(T, S, pc.s);
        if (app_run && lane < AB / 16) {
            const int which = lane / (D / 8), c = lane % (D / 8);
            cp_async16(ab_addr + lane * 16, (which ? a.v_new : a.k_new) + ((int64_t)pc.s * Hkv + pc.g) * D + c * 8);
        }
        if (pc.pe < u1) {  // the next piece's q rows
            const int s2 = find_seq(T, S, pc.pe);
            const int32_t nt2 = (T[s2 + 1] - T[s2]) / Hkv;
            const uint16_t *src = a.q + ((int64_t)s2 * Hq + (int64_t)((pc.pe - T[s2]) / nt2) * G) * D;
            for (uint32_t c = lane; c < QB / 16; c += 32) cp_async16(qb_addr + c * 16, src + c * 8);
        }
        cp_async_commit();
        for (int32_t uu = pc.pb; uu < pc.pe; ++uu) {
            const int st = (int)(consumed % kStages);
            const uint32_t par = (consumed / kStages) & 1u;
            uint8_t *Ks = k_of(st);
            uint8_t *Vs = Ks + TILE_BYTES;
            const uint32_t bk = bk_of(st), bv = bv_of(st);
            const int nvalid = min(kTile, pc.n - pc.skip - (uu - pc.run_begin) * kTile);
            const bool more = uu + kStages < u1;  // the unit this stage takes next
            const bool app = app_run && uu == pc.run_end - 1;
            const int arow = (pc.n - 1) % kTile;
            wait_phase(bk, par, a.err, dead);
            if (app) {
                cp_async_wait_all();  // the new K/V rows
                __syncwarp();
                if (lane < D / 8)
                    *reinterpret_cast<uint4 *>(Ks + swz(arow, lane)) = *reinterpret_cast<const uint4 *>(ab + lane * 16);
                __syncwarp();
            }
            comp.qk(Ks, nvalid);
            // the K stage is refilled by TMA next: order the warp's generic
            // shared-memory reads before the async-proxy write
            fence_proxy_async_smem();
            __syncwarp();
            if (more && lane == 0) issue_half<D>(&tmap, a, T, rows, cu0, uu + kStages, 0, smem_u32(Ks), bk, policy);
            wait_phase(bv, par, a.err, dead);
            if (app) {
                if (lane < D / 8)
                    *reinterpret_cast<uint4 *>(Vs + swz(arow, lane)) =
                        *reinterpret_cast<const uint4 *>(ab + D * 2 + lane * 16);
                __syncwarp();
            }
            comp.pv(Vs);
            if (app) {
                // store the new row into the pool: this warp's own TMA reads of
                // the tile have completed, and no other unit covers that row
                const int32_t k = uu - cu0;
                const int32_t y = k < a.rows_cap ? rows[k] : unit_row(a, T, uu);
                if (y >= 0 && lane < AB / 16) {
                    const int which = lane / (D / 8), c = lane % (D / 8);
                    const int64_t row = (int64_t)y + arow + (int64_t)which * Hkv * a.bs;
                    *reinterpret_cast<uint4 *>(a.pool + row * D + c * 8) =
                        *reinterpret_cast<const uint4 *>(ab + lane * 16);
                }
            }
            fence_proxy_async_smem();
            __syncwarp();
            if (more && lane == 0) issue_half<D>(&tmap, a, T, rows, cu0, uu + kStages, 1, smem_u32(Vs), bv, policy);
            ++consumed;
        }

        // ---- end of a piece: the output, or this part's partial ----
        const int32_t r = pc.s * Hkv + pc.g;
        const int32_t p_first = cta_of(pc.run_begin, W, NP);
        const int32_t p_last = cta_of(pc.run_end - 1, W, NP);
        // a run whose prefix lives in prefix records always leaves a partial
        const bool split = p_first != p_last || pc.skip > 0;
        uint16_t *orow = a.out + ((int64_t)pc.s * Hq + (int64_t)pc.g * G) * D;
        float *slot = a.ws_part + ((int64_t)r + part) * MF;
        make_ready();
        comp.store(orow, slot, split, lane);
        if (part == p_first && lane == 0)  // each run has one first part: it tells the combine
            a.ws_run[r] = make_int2(p_first, split ? p_last - p_first + 1 : 0);
        u = pc.pe;
    }
    if (chained) grid_dependency_wait();
}

// ------------------------------------------------------------ combine ---
// Split-K combine: for each (sequence, KV head) run cut by part boundaries
// (or with a shared prefix), merge its records (m_k, l_k, o_k) in order:
//     M = max_k m_k,  out = sum_k 2^(m_k - M) o_k / sum_k 2^(m_k - M) l_k
// (base-2 online-softmax state).  One CTA per run, covering all G*D output
// columns: NG thread groups of G*D/(4*CPT) threads (CPT float4 columns
// each) take records k = grp, grp + NG, ..., then merge their states in
// group order, so the result depends only on the run's shape.  Runs finished
// inside the attention kernel return at once.
struct CombineArgs {
    uint16_t *out;
    const int2 *ws_run;    // per run: (first part, parts), parts = 0 when not split
    const float *ws_part;
    int32_t S;
    int32_t Hkv;
    const int32_t *skip;   // cascade mode: sequences with skip > 0 also merge
    const float *ws_pre;   // KS prefix records [k][S][Hkv], ahead of their parts
    int32_t KS;
};

constexpr int kCombineMaxThreads = 1024;
constexpr int kCombineBatch = 8;  // records each thread loads per round trip

// Thread groups per combine CTA (a run's records are spread over the
// groups, kCombineBatch loads in flight per thread): enough groups for
// about 8 records per thread, up to 1024 threads, and at least 128 threads
// (one group when a run's output has 128 float4 columns or more).  Small
// CTAs leave room on the SMs for the next step's decode CTAs, which start
// as the combine's CTAs finish: on the Llama-3-8B-shaped layer (64
// sequences, 32 q / 8 KV heads) 128-thread CTAs took 54.5-54.9 µs per step
// against 55.1-55.4 with 256 (six same-box pairs), at a cost of about 1 µs
// in 296 for three co-located models, whose heavy-tailed runs take more
// round trips with one group.
template <int D, int G>
inline int combine_groups(double records_per_run, bool shared_prefix)
{
    constexpr int NC = G * D / 4;
    (void)shared_prefix;
    const int floor_threads = 128;
    const int base = NC >= floor_threads ? 1 : floor_threads / NC;
    const int most = kCombineMaxThreads / NC;
    int want = (int)(records_per_run / 8.0 + 0.999);
    return want < base ? base : (want > most ? most : want);
}

// Columns per thread CPT: 1, or 2 for the one-group form of shared-prefix
// mode.  There every member run is one CTA, and the agent chains have 2048
// of them: at one column a thread (128 threads a run) and 64 registers only
// eight CTAs fit an SM and the last 850 runs wait for a second wave; at two
// columns a thread (64 threads a run, registers held to 64, no shared
// memory) sixteen fit and one wave covers 2432 runs.  Each column merges the
// same records in the same order either way, so the bits do not change.
template <int D, int G, int CPT>
struct CombineShape {
    static constexpr int NC = G * D / 4;   // float4 columns of a run's output
    static constexpr int NCT = NC / CPT;   // threads of a group
    static constexpr int MAX_THREADS = CPT == 1 ? kCombineMaxThreads : NCT;
    static constexpr int MIN_CTAS = CPT == 1 ? 1 : 28 / ((NCT + 31) / 32);  // 28 warps an SM: 72 registers
    static constexpr int BATCH = CPT == 1 ? kCombineBatch : 4;
};

// shared memory of a CTA of `threads` threads: the groups' states for the
// in-order merge (none with one group)
template <int D, int G, int CPT>
inline size_t combine_smem_bytes(int threads)
{
    return threads > CombineShape<D, G, CPT>::NCT ? (size_t)threads * CPT * (2 * sizeof(float) + sizeof(float4)) : 0;
}

template <int D, int G, int CPT>
__global__ void __launch_bounds__(CombineShape<D, G, CPT>::MAX_THREADS, CombineShape<D, G, CPT>::MIN_CTAS)
combine_kernel(const __grid_constant__ CombineArgs c)
{
    using CS = CombineShape<D, G, CPT>;
    constexpr uint32_t MF = merge_floats<D, G>();
    constexpr int NCT = CS::NCT;
    constexpr int B = CS::BATCH;
    static_assert(CS::NC % CPT == 0 && NCT <= kCombineMaxThreads, "whole columns per thread");
    const int NG = (int)blockDim.x / NCT;  // groups of NCT threads
    extern __shared__ float4 s_dyn[];      // [CPT][blockDim] O, then M, then L (when NG > 1)
    const int r = blockIdx.x;
    grid_dependency_wait();  // the attention grid's partials and run table
    // Release the next grid only now, when every grid before this one has
    // completed: a decode grid that follows without a wait of its own (step
    // overlap) relies on it, and until its own wait writes nothing that this
    // grid reads or writes.
    grid_launch_dependents();
    const int2 info = c.ws_run[r];
    const int s = r / c.Hkv, g = r % c.Hkv;
    const int npre = (c.skip != nullptr && c.skip[s] > 0) ? c.KS : 0;
    const int cnt = info.y + npre;
    if (cnt == 0) return;  // finished inside the attention kernel (or empty)
    const float *base = c.ws_part + ((int64_t)r + info.x) * MF;
    uint16_t *orow = c.out + ((int64_t)s * c.Hkv * G + (int64_t)g * G) * D;
    const int tid = threadIdx.x;
    const int grp = tid / NCT;
    int col[CPT], h[CPT];
#pragma unroll
    for (int j = 0; j < CPT; ++j) {
        col[j] = tid % NCT + j * NCT;
        h[j] = (col[j] * 4) / D;
    }
    // online merge of this group's records per column: M running max, L and
    // O relative to M; records k = grp, grp + NG, ... are loaded B at a time
    float M[CPT], L[CPT];
    float4 O[CPT];
#pragma unroll
    for (int j = 0; j < CPT; ++j) {
        M[j] = -INFINITY;
        L[j] = 0.f;
        O[j] = make_float4(0.f, 0.f, 0.f, 0.f);
    }
    for (int k0 = grp; k0 < cnt; k0 += NG * B) {
        float mv[B][CPT], lv[B][CPT];
        float4 ov[B][CPT];
#pragma unroll
        for (int b = 0; b < B; ++b) {
            const int k = k0 + b * NG;
#pragma unroll
            for (int j = 0; j < CPT; ++j) mv[b][j] = -INFINITY;
            if (k < cnt) {
                const float *sl = k < npre ? c.ws_pre + (((int64_t)k * c.S + s) * c.Hkv + g) * MF
                                           : base + (int64_t)(k - npre) * MF;
#pragma unroll
                for (int j = 0; j < CPT; ++j) {
                    mv[b][j] = sl[G * D + h[j]];
                    lv[b][j] = sl[G * D + G + h[j]];
                    ov[b][j] = *reinterpret_cast<const float4 *>(sl + col[j] * 4);
                }
            }
        }
#pragma unroll
        for (int b = 0; b < B; ++b)
#pragma unroll
            for (int j = 0; j < CPT; ++j) {
                if (mv[b][j] == -INFINITY) continue;  // past the run's records
                const float Mn = fmaxf(M[j], mv[b][j]);
                const float sa = fast_exp2(M[j] - Mn), sb = fast_exp2(mv[b][j] - Mn);
                L[j] = L[j] * sa + lv[b][j] * sb;
                O[j].x = O[j].x * sa + ov[b][j].x * sb;
                O[j].y = O[j].y * sa + ov[b][j].y * sb;
                O[j].z = O[j].z * sa + ov[b][j].z * sb;
                O[j].w = O[j].w * sa + ov[b][j].w * sb;
                M[j] = Mn;
            }
    }
    if (NG > 1) {
        const int nt = (int)blockDim.x;
        float4 *s_O = s_dyn;
        float *s_M = reinterpret_cast<float *>(s_dyn + CPT * nt);
        float *s_L = s_M + CPT * nt;
#pragma unroll
        for (int j = 0; j < CPT; ++j) {
            s_M[j * nt + tid] = M[j];
            s_L[j * nt + tid] = L[j];
            s_O[j * nt + tid] = O[j];
        }
        __syncthreads();
        if (grp != 0) return;
        // merge the groups in order
        for (int q = 1; q < NG; ++q)
#pragma unroll
            for (int j = 0; j < CPT; ++j) {
                const int i = j * nt + tid + q * NCT;
                const float mq = s_M[i];
                if (mq == -INFINITY) continue;  // group had no records
                const float Mn = fmaxf(M[j], mq);
                const float sa = fast_exp2(M[j] - Mn), sb = fast_exp2(mq - Mn);
                const float4 oq = s_O[i];
                L[j] = L[j] * sa + s_L[i] * sb;
                O[j].x = O[j].x * sa + oq.x * sb;
                O[j].y = O[j].y * sa + oq.y * sb;
                O[j].z = O[j].z * sa + oq.z * sb;
                O[j].w = O[j].w * sa + oq.w * sb;
                M[j] = Mn;
            }
    }
#pragma unroll
    for (int j = 0; j < CPT; ++j) {
        __nv_bfloat162 lo = __floats2bfloat162_rn(O[j].x / L[j], O[j].y / L[j]);
        __nv_bfloat162 hi = __floats2bfloat162_rn(O[j].z / L[j], O[j].w / L[j]);
        uint2 w2;
        w2.x = *reinterpret_cast<uint32_t *>(&lo);
        w2.y = *reinterpret_cast<uint32_t *>(&hi);
        *reinterpret_cast<uint2 *>(orow + col[j] * 4) = w2;
    }
}

// host helpers ---------------------------------------------------------------
constexpr int kRowsCap = 2048;

template <int D, int G>
inline size_t attn_smem_bytes(int S, int rows_cap, int nwarps)
{
    const size_t stage = 2ull * (D / 64) * kHalfBytes;
    const size_t bufs = (size_t)G * D * 2 + 2 * D * 2;  // per warp: q rows, new K/V rows
    return 1024 + (size_t)nwarps * (kStages * stage + bufs) + (2 * nwarps * kStages) * 8 + 64 + (size_t)(3 * S + 1) * 4 +
           (size_t)rows_cap * 4;
}

// partial records: one per (run, part) pair that a run can touch (parts:
// at most kWarps per CTA)
inline size_t attn_partial_slots(int S, int Hkv, int P) { return (size_t)S * Hkv + (size_t)P * kWarps; }

}  // namespace kvp
