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
//   CTA i of P processes the contiguous unit range [i*W/P, (i+1)*W/P): every
//           CTA streams the same number of bytes (+-1 tile) whatever the
//           length distribution.
//   piece = the part of one run inside one CTA's range.  A run covered by
//           one CTA is finished in place; a run cut by CTA boundaries leaves
//           one fp32 partial (max, sum, unnormalised output) per CTA, and the
//           last CTA to arrive (per-run counter) merges them in CTA order.
// Inside a CTA each of the 4 warps owns every 4th unit of a piece and a
// private ring of shared-memory stages fed by 2-D TMA loads (128-byte
// swizzle) that run ahead across piece boundaries.  The 4 warps' states are
// merged through shared memory at the end of a piece.
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

constexpr int kWarps = 4;
constexpr int kThreads = kWarps * 32;
constexpr int kTile = 16;              // tokens per unit
constexpr uint32_t kHalfBytes = kTile * 128;  // one 64-column box: 16 rows x 128 B
constexpr uint64_t kWaitLimitNs = 2000000000ull;  // bounded mbarrier waits: 2 s

struct AttnArgs {
    const uint16_t *q;
    uint16_t *out;
    const int32_t *table;
    const int32_t *ctx_lens;
    int32_t *err;
    float *ws_part;
    int32_t *ws_cnt;
    int64_t rows_per_page;   // page_bytes / (d * 2)
    int64_t pool_pages;
    int32_t pages_per_block;
    int32_t max_blocks;
    int32_t S;
    int32_t Hkv;
    int32_t bs;
    int32_t nsw;             // stages per warp
    int32_t P;               // CTAs (work partitions)
    float qk_scale;          // scale * log2(e)
};

__device__ __forceinline__ void report(int32_t *err, int code) { atomicCAS(err, 0, code); }

// bounded wait on an mbarrier phase; a wait that exceeds the limit records
// KV_ERR_DEVICE_TIMEOUT and makes every later wait of this warp return at once
__device__ __forceinline__ void wait_stage(uint32_t bar, uint32_t parity, int32_t *err, bool &dead)
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
    int grp, sub;

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

    __device__ __forceinline__ void tile(const uint8_t *Ks, const uint8_t *Vs, int nvalid)
    {
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
                sc[i][h] = fast_exp2(sc[i][h] - m[h]);
                l[h] += sc[i][h];
            }
#pragma unroll
        for (int i = 0; i < TPG; ++i) {
            const int t = grp + i * NGRP;
            if (t < nvalid) {
#pragma unroll
                for (int j = 0; j < NCH; ++j) {
                    uint4 w = *reinterpret_cast<const uint4 *>(Vs + swz(t, sub + j * LPT));
                    uint32_t ws[4] = {w.x, w.y, w.z, w.w};
#pragma unroll
                    for (int e = 0; e < 4; ++e) {
                        float2 vv = make_float2(bf_lo(ws[e]), bf_hi(ws[e]));
#pragma unroll
                        for (int h = 0; h < G; ++h)
                            o[h][j * 4 + e] = __ffma2_rn(make_float2(sc[i][h], sc[i][h]), vv, o[h][j * 4 + e]);
                    }
                }
            }
        }
    }

    // write this warp's (o[G][D], m[G], l[G]) to shared memory
    __device__ __forceinline__ void finish(float *mw, int lane)
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
                    float4 *dst = reinterpret_cast<float4 *>(mw + h * D + c * 8);
                    dst[0] = make_float4(o[h][j * 4 + 0].x, o[h][j * 4 + 0].y, o[h][j * 4 + 1].x, o[h][j * 4 + 1].y);
                    dst[1] = make_float4(o[h][j * 4 + 2].x, o[h][j * 4 + 2].y, o[h][j * 4 + 3].x, o[h][j * 4 + 3].y);
                }
        }
        if (lane == 0) {
#pragma unroll
            for (int h = 0; h < G; ++h) {
                mw[G * D + h] = m[h];
                mw[G * D + G + h] = l[h];
            }
        }
    }
};

// ----------------------------------------------------------- tensor cores --
template <int D, int G>
struct MmaCompute {
    static_assert(G <= 8, "query-head group must fit the n=8 MMA tile");
    static constexpr int KS = D / 16;
    uint32_t qf[KS][2];  // B operand of q.K: Q^T fragments (bf16x2)
    float acc[KS][4];    // O^T accumulators, 16 d-rows per block
    float m[2], l[2];    // heads 2*tig, 2*tig+1
    float qk_scale;
    int gid, tig, lane_;

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

    __device__ __forceinline__ void tile(const uint8_t *Ks, uint8_t *Vs, int nvalid)
    {
        // rows past the context may hold anything (even NaN bit patterns);
        // P is zero there, but 0 * NaN is NaN inside the MMA, so clear them
        if (nvalid < kTile) {
            const int nchunk = (kTile - nvalid) * (D / 8);
            for (int idx = lane_; idx < nchunk; idx += 32) {
                const int r = nvalid + idx / (D / 8);
                const int c = idx % (D / 8);
                *reinterpret_cast<uint4 *>(Vs + swz(r, c)) = make_uint4(0u, 0u, 0u, 0u);
            }
            __syncwarp();
        }
        const uint32_t kbase = smem_u32(Ks);
        const uint32_t vbase = smem_u32(Vs);
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
        float x0 = ok0 ? s[0] * qk_scale : -INFINITY;
        float x1 = ok0 ? s[1] * qk_scale : -INFINITY;
        float x2 = ok1 ? s[2] * qk_scale : -INFINITY;
        float x3 = ok1 ? s[3] * qk_scale : -INFINITY;
        float t0 = fmaxf(x0, x2), t1 = fmaxf(x1, x3);
#pragma unroll
        for (int off = 4; off < 32; off <<= 1) {
            t0 = fmaxf(t0, __shfl_xor_sync(0xffffffffu, t0, off));
            t1 = fmaxf(t1, __shfl_xor_sync(0xffffffffu, t1, off));
        }
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
        const uint32_t b0 = movmatrix_trans(*reinterpret_cast<uint32_t *>(&lo));
        const uint32_t b1 = movmatrix_trans(*reinterpret_cast<uint32_t *>(&hi));
#pragma unroll
        for (int mb = 0; mb < KS; ++mb) {
            uint32_t a0, a1, a2, a3;
            ldmatrix_x4_trans(vbase + swz(r8 + (mat >> 1) * 8, mb * 2 + (mat & 1)), a0, a1, a2, a3);
            mma_bf16_16816(acc[mb], a0, a1, a2, a3, b0, b1);
        }
    }

    __device__ __forceinline__ void finish(float *mw, int lane)
    {
#pragma unroll
        for (int off = 4; off < 32; off <<= 1) {
            l[0] += __shfl_xor_sync(0xffffffffu, l[0], off);
            l[1] += __shfl_xor_sync(0xffffffffu, l[1], off);
        }
        const int h0 = 2 * tig, h1 = 2 * tig + 1;
#pragma unroll
        for (int mb = 0; mb < KS; ++mb) {
            const int d0 = mb * 16 + gid;
            if (h0 < G) {
                mw[h0 * D + d0] = acc[mb][0];
                mw[h0 * D + d0 + 8] = acc[mb][2];
            }
            if (h1 < G) {
                mw[h1 * D + d0] = acc[mb][1];
                mw[h1 * D + d0 + 8] = acc[mb][3];
            }
        }
        if (gid == 0) {
            if (h0 < G) {
                mw[G * D + h0] = m[0];
                mw[G * D + G + h0] = l[0];
            }
            if (h1 < G) {
                mw[G * D + h1] = m[1];
                mw[G * D + G + h1] = l[1];
            }
        }
        (void)lane;
    }
};

// ---------------------------------------------------------------- stream ---
// Walks one warp's units across the pieces of its CTA's range: within a piece
// [pb, pe) the warp owns units pb + warp, pb + warp + 4, ...
struct Piece {
    int32_t pb, pe;        // piece unit range
    int32_t run_begin;     // unit id of tile 0 of this (s, g) run
    int32_t run_end;
    int32_t s, g, n;       // sequence, KV head, context length
};

__device__ __forceinline__ int32_t clamp_len(const AttnArgs &a, int s, bool report_errors)
{
    int32_t n = a.ctx_lens[s];
    const int32_t cap = a.max_blocks * a.bs;
    if (n < 0 || n > cap) {
        if (report_errors) report(a.err, KV_ERR_DEVICE_BOUNDS);
        n = n < 0 ? 0 : cap;
    }
    return n;
}

// T[s] = first unit of sequence s (T[S] = total); find the run holding u
__device__ __forceinline__ void decode_piece(const AttnArgs &a, const int32_t *T, int32_t u, int32_t u1, Piece &p)
{
    int lo = 0, hi = a.S;  // largest s with T[s] <= u (T is non-decreasing)
    while (hi - lo > 1) {
        const int mid = (lo + hi) >> 1;
        if (T[mid] <= u) lo = mid; else hi = mid;
    }
    const int s = lo;
    const int32_t nt = (T[s + 1] - T[s]) / a.Hkv;
    const int32_t g = (u - T[s]) / nt;
    p.s = s;
    p.g = g;
    p.n = clamp_len(a, s, false);
    p.run_begin = T[s] + g * nt;
    p.run_end = p.run_begin + nt;
    p.pb = u;
    p.pe = p.run_end < u1 ? p.run_end : u1;
}

struct Producer {
    Piece p;
    int32_t u;   // next unit to load
    int32_t u1;
    bool valid;

    __device__ __forceinline__ void normalise(const AttnArgs &a, const int32_t *T, int warp)
    {
        while (valid && u >= p.pe) {
            if (p.pe >= u1) {
                valid = false;
                break;
            }
            decode_piece(a, T, p.pe, u1, p);
            u = p.pb + warp;
        }
    }
    __device__ __forceinline__ void start(const AttnArgs &a, const int32_t *T, int32_t u0, int32_t uend, int warp)
    {
        u1 = uend;
        valid = u0 < uend;
        if (!valid) return;
        decode_piece(a, T, u0, u1, p);
        u = p.pb + warp;
        normalise(a, T, warp);
    }
    __device__ __forceinline__ void advance(const AttnArgs &a, const int32_t *T, int warp)
    {
        u += kWarps;
        normalise(a, T, warp);
    }
};

template <int D>
__device__ __forceinline__ void issue_unit(const CUtensorMap *tmap, const AttnArgs &a, const Producer &pr,
                                           uint32_t stage_addr, uint32_t bar, uint64_t policy)
{
    constexpr int HALVES = D / 64;
    constexpr uint32_t TILE_BYTES = HALVES * kHalfBytes;
    const int32_t tile = pr.u - pr.p.run_begin;
    const int32_t tok0 = tile * kTile;
    const int32_t lb = tok0 / a.bs;
    const int32_t phys = a.table[(int64_t)pr.p.s * a.max_blocks + lb];
    if (phys < 0 || (int64_t)phys + a.pages_per_block > a.pool_pages) {
        report(a.err, KV_ERR_DEVICE_BOUNDS);
        mbar_arrive(bar);  // complete the phase without data
        return;
    }
    const int64_t row0 = (int64_t)phys * a.rows_per_page + (tok0 % a.bs);
    const int32_t yk = (int32_t)(row0 + (int64_t)pr.p.g * a.bs);
    const int32_t yv = (int32_t)(row0 + (int64_t)(a.Hkv + pr.p.g) * a.bs);
    mbar_arrive_expect_tx(bar, 2 * TILE_BYTES);
#pragma unroll
    for (int h = 0; h < HALVES; ++h) {
        tma_load_2d(stage_addr + h * kHalfBytes, tmap, h * 64, yk, bar, policy);
        tma_load_2d(stage_addr + TILE_BYTES + h * kHalfBytes, tmap, h * 64, yv, bar, policy);
    }
}

// first CTA whose range contains unit u
__device__ __forceinline__ int32_t cta_of(int64_t u, int64_t W, int64_t P)
{
    return (int32_t)(((u + 1) * P - 1) / W);
}

// per-warp merge record and per-CTA partial: o[G][D], m[G], l[G], padded to
// a multiple of 4 floats so every record starts 16-byte aligned
template <int D, int G>
__host__ __device__ constexpr uint32_t merge_floats() { return (G * D + 2 * G + 3) / 4 * 4; }

template <int D, int G, class Comp>
__global__ void __launch_bounds__(kThreads, 1)
paged_attn_kernel(const __grid_constant__ CUtensorMap tmap, const __grid_constant__ AttnArgs a)
{
    constexpr int HALVES = D / 64;
    constexpr uint32_t TILE_BYTES = HALVES * kHalfBytes;
    constexpr uint32_t STAGE_BYTES = 2 * TILE_BYTES;
    constexpr uint32_t MF = merge_floats<D, G>();
    extern __shared__ uint8_t smem_raw[];
    // stages need 1024-byte alignment for the 128-byte swizzle pattern
    uint8_t *smem = smem_raw + ((1024u - (smem_u32(smem_raw) & 1023u)) & 1023u);
    const int nsw = a.nsw;
    uint8_t *stages = smem;
    float *merge = reinterpret_cast<float *>(smem + (size_t)kWarps * nsw * STAGE_BYTES);
    uint64_t *bars = reinterpret_cast<uint64_t *>(merge + kWarps * MF);
    int32_t *misc = reinterpret_cast<int32_t *>(bars + kWarps * nsw);  // [0..7] scratch
    int32_t *T = misc + 8;                                              // [S + 1]

    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int S = a.S, Hkv = a.Hkv, Hq = a.Hkv * G;

    if (tid == 0) {
        for (int i = 0; i < kWarps * nsw; ++i) mbar_init(smem_u32(&bars[i]), 1);
        fence_mbar_init();
    }
    if (tid == 32) prefetch_tensormap(&tmap);

    // ---- prologue: T[s] = first unit of sequence s ----
    {
        const int per = (S + kThreads - 1) / kThreads;
        const int lo = min(S, tid * per), hi = min(S, lo + per);
        int32_t local = 0;
        for (int s = lo; s < hi; ++s) {
            const int32_t n = clamp_len(a, s, true);
            local += ((n + kTile - 1) / kTile) * Hkv;
            if (n == 0 && (s % a.P) == (int)blockIdx.x) {
                // an empty context has no softmax: its output is defined as zero
                for (int i = 0; i < Hq * D; ++i) a.out[(int64_t)s * Hq * D + i] = 0;
            }
        }
        // block exclusive scan of `local`
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
        for (int s = lo; s < hi; ++s) {
            T[s] = run;
            run += ((clamp_len(a, s, false) + kTile - 1) / kTile) * Hkv;
        }
        if (tid == 0) {
            int32_t tot = 0;
            for (int w = 0; w < kWarps; ++w) tot += misc[w];
            T[S] = tot;
        }
        __syncthreads();
    }

    // with fewer units than CTAs only the first W CTAs take work, so that
    // every working CTA's range is non-empty and a run's contributors are
    // exactly the CTAs cta_of(first unit) .. cta_of(last unit)
    const int64_t W = T[S];
    const int64_t P = W < (int64_t)a.P ? W : (int64_t)a.P;
    if ((int64_t)blockIdx.x >= P) return;
    const int32_t u0 = (int32_t)((int64_t)blockIdx.x * W / P);
    const int32_t u1 = (int32_t)((int64_t)(blockIdx.x + 1) * W / P);
    if (u0 >= u1) return;  // no units for this CTA (no barriers are shared beyond here)

    const uint64_t policy = l2_policy_evict_first();
    uint8_t *my_stages = stages + (size_t)warp * nsw * STAGE_BYTES;
    uint64_t *my_bars = bars + warp * nsw;

    Producer pr;
    pr.start(a, T, u0, u1, warp);
    for (int k = 0; k < nsw && pr.valid; ++k) {
        if (lane == 0) issue_unit<D>(&tmap, a, pr, smem_u32(my_stages + k * STAGE_BYTES), smem_u32(&my_bars[k]), policy);
        pr.advance(a, T, warp);
    }

    bool dead = false;
    uint32_t consumed = 0;
    int32_t u = u0;
    while (u < u1) {
        Piece pc;
        decode_piece(a, T, u, u1, pc);
        Comp comp;
        comp.begin(a.q + ((int64_t)pc.s * Hq + (int64_t)pc.g * G) * D, a.qk_scale, lane);
        for (int32_t uu = pc.pb + warp; uu < pc.pe; uu += kWarps) {
            const uint32_t st = consumed % (uint32_t)nsw;
            wait_stage(smem_u32(&my_bars[st]), (consumed / (uint32_t)nsw) & 1u, a.err, dead);
            uint8_t *Ks = my_stages + st * STAGE_BYTES;
            const int32_t tok0 = (uu - pc.run_begin) * kTile;
            const int nvalid = min(kTile, pc.n - tok0);
            comp.tile(Ks, Ks + TILE_BYTES, nvalid);
            // this stage is refilled by TMA next: order the warp's generic
            // shared-memory accesses before the async-proxy write
            fence_proxy_async_smem();
            __syncwarp();
            if (pr.valid) {
                if (lane == 0) {
                    issue_unit<D>(&tmap, a, pr, smem_u32(Ks), smem_u32(&my_bars[st]), policy);
                }
                pr.advance(a, T, warp);
            }
            ++consumed;
        }
        comp.finish(merge + warp * MF, lane);
        __syncthreads();

        // ---- merge the 4 warps; finish the run or leave a partial ----
        const int32_t r = pc.s * Hkv + pc.g;
        const int32_t i_first = cta_of(pc.run_begin, W, P);
        const int32_t i_last = cta_of(pc.run_end - 1, W, P);
        const bool split = i_first != i_last;
        float *slot = a.ws_part + (int64_t)(r + (int32_t)blockIdx.x) * MF;
        uint16_t *orow = a.out + ((int64_t)pc.s * Hq + (int64_t)pc.g * G) * D;
        for (int idx = tid; idx < G * D; idx += kThreads) {
            const int h = idx / D;
            float M = -INFINITY;
#pragma unroll
            for (int w = 0; w < kWarps; ++w) M = fmaxf(M, merge[w * MF + G * D + h]);
            float L = 0.f, O = 0.f;
#pragma unroll
            for (int w = 0; w < kWarps; ++w) {
                const float sc = fast_exp2(merge[w * MF + G * D + h] - M);
                L += sc * merge[w * MF + G * D + G + h];
                O += sc * merge[w * MF + idx];
            }
            if (!split) {
                orow[idx] = __bfloat16_as_ushort(__float2bfloat16_rn(O / L));
            } else {
                slot[idx] = O;
                if (idx % D == 0) {
                    slot[G * D + h] = M;
                    slot[G * D + G + h] = L;
                }
            }
        }
        if (split) {
            __threadfence();
            __syncthreads();
            if (tid == 0) {
                const int32_t prev = atomicAdd(&a.ws_cnt[r], 1);
                const int last = prev == i_last - i_first;
                if (last) atomicExch(&a.ws_cnt[r], 0);
                misc[4] = last;
            }
            __syncthreads();
            if (misc[4]) {
                __threadfence();
                const float *base = a.ws_part + (int64_t)(r + i_first) * MF;
                const int cnt = i_last - i_first + 1;
                for (int idx = tid; idx < G * D; idx += kThreads) {
                    const int h = idx / D;
                    float M = -INFINITY;
                    for (int k = 0; k < cnt; ++k) M = fmaxf(M, __ldcg(base + (int64_t)k * MF + G * D + h));
                    float L = 0.f, O = 0.f;
                    for (int k = 0; k < cnt; ++k) {
                        const float *sl = base + (int64_t)k * MF;
                        const float sc = fast_exp2(__ldcg(sl + G * D + h) - M);
                        L += sc * __ldcg(sl + G * D + G + h);
                        O += sc * __ldcg(sl + idx);
                    }
                    orow[idx] = __bfloat16_as_ushort(__float2bfloat16_rn(O / L));
                }
            }
        }
        __syncthreads();
        u = pc.pe;
    }
}

// host helpers ---------------------------------------------------------------
template <int D, int G>
inline size_t attn_smem_bytes(int nsw, int S)
{
    const size_t stage = 2ull * (D / 64) * kHalfBytes;
    return 1024 + (size_t)kWarps * nsw * stage + (size_t)kWarps * merge_floats<D, G>() * 4 +
           (size_t)kWarps * nsw * 8 + 32 + (size_t)(S + 1) * 4;
}

}  // namespace kvp
