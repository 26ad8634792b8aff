// cascade_impl.cuh -- shared-prefix ("cascade") attention for sequences whose
// block tables start with the same physical blocks.
//
// Sequences that share a prefix by reference (agent stages building on one
// system prompt, §III-B / §III-C) hold identical K/V for its tokens, so the
// prefix's contribution to every sharer's decode query is one dense
// contraction per KV head: all sharers' query heads of that KV head form the
// rows, the prefix tokens the columns.  The prefix K/V is then read once per
// (row tile, key split) from L2 instead of once per sharer, and the work runs
// on the tensor cores as a small flash-attention forward:
//   S = Q K^T (m16n8k16 bf16 -> fp32), online softmax in base 2,
//   O += P V, per 64-key tile streamed through a 3-stage TMA pipeline.
// Each CTA leaves, per (sharer, KV head), one fp32 record (unnormalised o,
// running max m, sum l) in the same format as the decode kernel's split
// partials; the combine kernel merges prefix and suffix records, which is
// exact because the softmax over the whole context factorises over any
// partition of the keys.
#pragma once

#include "attn_impl.cuh"

namespace kvp {

constexpr int kPreWarps = 4;
constexpr int kPreThreads = kPreWarps * 32;
constexpr int kPreRows = kPreWarps * 16;  // query rows (sharer, head) per CTA
constexpr int kPreKeys = 64;              // prefix tokens per pipeline tile
constexpr int kPreStages = 3;
constexpr int kPreRowsCap = 1024;         // 16-token sub-tiles resolved up front
constexpr int kMaxKeySplits = 8;
constexpr int kCascadeWords = 4080;       // plan words carried as kernel parameters

struct CascadeArgs {
    const uint16_t *q;
    const int32_t *table;
    int32_t *err;
    float *ws_pre;        // [kMaxKeySplits][S][Hkv] records of merge_floats<D, G>() floats
    int32_t *ws_skip;     // [S]: shared-prefix tokens per sequence (0 = none)
    int64_t rows_per_page;
    int64_t pool_pages;
    int32_t pages_per_block;
    int32_t max_blocks;
    int32_t S;
    int32_t Hkv;
    int32_t bs;
    int32_t KS;           // key splits of every group's prefix
    int32_t n_groups;
    int32_t n_members;
    float qk_scale;       // scale * log2(e)
    int32_t pad;
    // [n_groups + 1] first row tile of each group | [n_groups + 1] first member
    // index | [n_groups] prefix tokens | [n_members] member sequences | [S] skip
    int32_t data[kCascadeWords];
};

// rows per row tile: whole query-head groups of consecutive members
template <int G>
__host__ __device__ constexpr int pre_members_per_tile() { return kPreRows / G; }

// Pool row (TMA y) of the K sub-tile holding prefix tokens 16q .. 16q+15 for
// KV head g, read from the lead member's table; -1 if outside the pool.
__device__ __forceinline__ int32_t pre_sub_row(const CascadeArgs &c, int lead, int g, int32_t q)
{
    const int32_t tok = q * kTile;
    const int32_t phys = c.table[(int64_t)lead * c.max_blocks + tok / c.bs];
    if (phys < 0 || (int64_t)phys + c.pages_per_block > c.pool_pages) return -1;
    return (int32_t)((int64_t)phys * c.rows_per_page + (int64_t)g * c.bs + tok % c.bs);
}

__device__ __forceinline__ uint32_t pack_bf16(float lo, float hi)
{
    __nv_bfloat162 v = __floats2bfloat162_rn(lo, hi);
    return *reinterpret_cast<uint32_t *>(&v);
}

template <int D, int G>
__global__ void __launch_bounds__(kPreThreads)
cascade_prefix_kernel(const __grid_constant__ CUtensorMap tmap, const __grid_constant__ CascadeArgs c)
{
    constexpr int HALVES = D / 64;
    constexpr uint32_t SUB_BYTES = HALVES * kHalfBytes;           // 16 tokens x D
    constexpr uint32_t KT_BYTES = (kPreKeys / kTile) * SUB_BYTES;  // 64 tokens x D
    constexpr uint32_t STAGE_BYTES = 2 * KT_BYTES;                 // K then V
    constexpr uint32_t MF = merge_floats<D, G>();
    constexpr int MT = pre_members_per_tile<G>();
    constexpr int KSL = D / 16;        // k-slices of q.K
    constexpr int NT = kPreKeys / 8;   // key n-tiles of S
    constexpr int ND = D / 8;          // d n-tiles of O
    extern __shared__ uint8_t smem_raw[];
    uint8_t *smem = smem_raw + ((1024u - (smem_u32(smem_raw) & 1023u)) & 1023u);
    uint64_t *bars = reinterpret_cast<uint64_t *>(smem + kPreStages * STAGE_BYTES);
    int32_t *rows = reinterpret_cast<int32_t *>(bars + kPreStages);  // [kPreRowsCap]

    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int gid = lane >> 2, tig = lane & 3;
    int bid = blockIdx.x;
    const int ks = bid % c.KS;
    bid /= c.KS;
    const int g = bid % c.Hkv;
    const int tile = bid / c.Hkv;

    const int32_t *tile_off = c.data;
    const int32_t *mem_off = tile_off + c.n_groups + 1;
    const int32_t *tokens = mem_off + c.n_groups + 1;
    const int32_t *members = tokens + c.n_groups;
    const int32_t *skip = members + c.n_members;
    int grp = 0;
    while (grp + 1 < c.n_groups && tile_off[grp + 1] <= tile) ++grp;
    const int m0 = mem_off[grp] + (tile - tile_off[grp]) * MT;  // this tile's members [m0, m1)
    const int m1 = min(m0 + MT, mem_off[grp + 1]);
    const int lead = members[mem_off[grp]];
    const int kt_all = tokens[grp] / kPreKeys;
    const int kt0 = ks * kt_all / c.KS, kt1 = (ks + 1) * kt_all / c.KS;  // non-empty: KS <= kt_all
    const int nkt = kt1 - kt0;

    if (tid == 0) {
        for (int i = 0; i < kPreStages; ++i) mbar_init(smem_u32(&bars[i]), 1);
        fence_mbar_init();
    }
    if (tid == 32) prefetch_tensormap(&tmap);
    grid_launch_dependents();
    grid_dependency_wait();  // the table (and q) come from the grids before

    if (blockIdx.x == 0)
        for (int s = tid; s < c.S; s += kPreThreads) c.ws_skip[s] = skip[s];
    const int nsub = nkt * (kPreKeys / kTile);
    for (int i = tid; i < min(nsub, kPreRowsCap); i += kPreThreads)
        rows[i] = pre_sub_row(c, lead, g, kt0 * (kPreKeys / kTile) + i);
    __syncthreads();

    // K and V of key tile i (relative to kt0) into stage st; thread 0 only
    auto issue = [&](int st, int i) {
        const uint32_t kdst = smem_u32(smem + st * STAGE_BYTES), vdst = kdst + KT_BYTES;
        const uint32_t bar = smem_u32(&bars[st]);
        int32_t y[kPreKeys / kTile];
        bool ok = true;
#pragma unroll
        for (int j = 0; j < kPreKeys / kTile; ++j) {
            const int32_t q = i * (kPreKeys / kTile) + j;
            y[j] = q < kPreRowsCap ? rows[q] : pre_sub_row(c, lead, g, kt0 * (kPreKeys / kTile) + q);
            ok = ok && y[j] >= 0;
        }
        if (!ok) {
            report(c.err, KV_ERR_DEVICE_BOUNDS);
            mbar_arrive(bar);  // complete the phase without data
            return;
        }
        const uint64_t pol = l2_policy_evict_normal();  // the prefix is re-read by every row tile
        mbar_arrive_expect_tx(bar, STAGE_BYTES);
#pragma unroll
        for (int j = 0; j < kPreKeys / kTile; ++j)
#pragma unroll
            for (int h = 0; h < HALVES; ++h) {
                const uint32_t off = j * SUB_BYTES + h * kHalfBytes;
                tma_load_2d(kdst + off, &tmap, h * 64, y[j], bar, pol);
                tma_load_2d(vdst + off, &tmap, h * 64, y[j] + c.Hkv * c.bs, bar, pol);
            }
    };
    if (tid == 0)
        for (int i = 0; i < kPreStages && i < nkt; ++i) issue(i, i);

    // Q fragments (A operand, row-major 16 x 16 per k-slice) straight from global
    const int r0 = warp * 16 + gid, r1 = r0 + 8;
    const int mi0 = m0 + r0 / G, mi1 = m0 + r1 / G;
    const bool v0 = r0 < MT * G && mi0 < m1, v1 = r1 < MT * G && mi1 < m1;
    const int Hq = c.Hkv * G;
    const uint16_t *q0 = v0 ? c.q + ((int64_t)members[mi0] * Hq + (int64_t)g * G + r0 % G) * D : nullptr;
    const uint16_t *q1 = v1 ? c.q + ((int64_t)members[mi1] * Hq + (int64_t)g * G + r1 % G) * D : nullptr;
    uint32_t qa[KSL][4];
#pragma unroll
    for (int kk = 0; kk < KSL; ++kk) {
        const int col = kk * 16 + 2 * tig;
        qa[kk][0] = v0 ? *reinterpret_cast<const uint32_t *>(q0 + col) : 0u;
        qa[kk][1] = v1 ? *reinterpret_cast<const uint32_t *>(q1 + col) : 0u;
        qa[kk][2] = v0 ? *reinterpret_cast<const uint32_t *>(q0 + col + 8) : 0u;
        qa[kk][3] = v1 ? *reinterpret_cast<const uint32_t *>(q1 + col + 8) : 0u;
    }

    float o[ND][4];
#pragma unroll
    for (int nd = 0; nd < ND; ++nd) o[nd][0] = o[nd][1] = o[nd][2] = o[nd][3] = 0.f;
    float mr0 = -INFINITY, mr1 = -INFINITY, l0 = 0.f, l1 = 0.f;
    bool dead = false;

    for (int i = 0; i < nkt; ++i) {
        const int st = i % kPreStages;
        wait_phase(smem_u32(&bars[st]), (uint32_t)(i / kPreStages) & 1u, c.err, dead);
        const uint32_t kb = smem_u32(smem + st * STAGE_BYTES), vb = kb + KT_BYTES;
        if (!dead) {
            // ---- S = Q K^T over 64 keys ----
            float s[NT][4];
#pragma unroll
            for (int nt = 0; nt < NT; ++nt) s[nt][0] = s[nt][1] = s[nt][2] = s[nt][3] = 0.f;
#pragma unroll
            for (int kk = 0; kk < KSL; ++kk)
#pragma unroll
                for (int nt = 0; nt < NT; nt += 2) {
                    const int key = (nt + (lane >> 4)) * 8 + (lane & 7);
                    const int chunk = 2 * kk + ((lane >> 3) & 1);
                    uint32_t b0, b1, b2, b3;
                    ldmatrix_x4(kb + (key >> 4) * SUB_BYTES + swz(key & 15, chunk), b0, b1, b2, b3);
                    mma_bf16_16816(s[nt], qa[kk][0], qa[kk][1], qa[kk][2], qa[kk][3], b0, b1);
                    mma_bf16_16816(s[nt + 1], qa[kk][0], qa[kk][1], qa[kk][2], qa[kk][3], b2, b3);
                }
            // ---- online softmax (base 2): rows r0 (c0, c1) and r1 (c2, c3) ----
            float t0 = -INFINITY, t1 = -INFINITY;
#pragma unroll
            for (int nt = 0; nt < NT; ++nt) {
                s[nt][0] *= c.qk_scale;
                s[nt][1] *= c.qk_scale;
                s[nt][2] *= c.qk_scale;
                s[nt][3] *= c.qk_scale;
                t0 = fmaxf(t0, fmaxf(s[nt][0], s[nt][1]));
                t1 = fmaxf(t1, fmaxf(s[nt][2], s[nt][3]));
            }
#pragma unroll
            for (int off = 1; off < 4; off <<= 1) {
                t0 = fmaxf(t0, __shfl_xor_sync(0xffffffffu, t0, off));
                t1 = fmaxf(t1, __shfl_xor_sync(0xffffffffu, t1, off));
            }
            const float mn0 = fmaxf(mr0, t0), mn1 = fmaxf(mr1, t1);
            const float a0 = fast_exp2(mr0 - mn0), a1 = fast_exp2(mr1 - mn1);
            mr0 = mn0;
            mr1 = mn1;
            l0 *= a0;
            l1 *= a1;
#pragma unroll
            for (int nd = 0; nd < ND; ++nd) {
                o[nd][0] *= a0;
                o[nd][1] *= a0;
                o[nd][2] *= a1;
                o[nd][3] *= a1;
            }
            uint32_t pa[NT / 2][4];  // P as A operand, one 16-key slice per entry
#pragma unroll
            for (int nt = 0; nt < NT; ++nt) {
                const float p0 = fast_exp2(s[nt][0] - mn0), p1 = fast_exp2(s[nt][1] - mn0);
                const float p2 = fast_exp2(s[nt][2] - mn1), p3 = fast_exp2(s[nt][3] - mn1);
                l0 += p0 + p1;
                l1 += p2 + p3;
                pa[nt >> 1][(nt & 1) * 2 + 0] = pack_bf16(p0, p1);
                pa[nt >> 1][(nt & 1) * 2 + 1] = pack_bf16(p2, p3);
            }
            // ---- O += P V ----
#pragma unroll
            for (int j = 0; j < NT / 2; ++j)
#pragma unroll
                for (int nd = 0; nd < ND; nd += 2) {
                    const int key = 16 * j + ((lane >> 3) & 1) * 8 + (lane & 7);
                    const int chunk = nd + (lane >> 4);
                    uint32_t b0, b1, b2, b3;
                    ldmatrix_x4_trans(vb + (key >> 4) * SUB_BYTES + swz(key & 15, chunk), b0, b1, b2, b3);
                    mma_bf16_16816(o[nd], pa[j][0], pa[j][1], pa[j][2], pa[j][3], b0, b1);
                    mma_bf16_16816(o[nd + 1], pa[j][0], pa[j][1], pa[j][2], pa[j][3], b2, b3);
                }
        }
        // every warp is done with this stage: refill it with tile i + stages
        fence_proxy_async_smem();
        __syncthreads();
        if (tid == 0 && i + kPreStages < nkt) issue(st, i + kPreStages);
    }

    // ---- this CTA's record per (sharer, KV head) ----
#pragma unroll
    for (int off = 1; off < 4; off <<= 1) {
        l0 += __shfl_xor_sync(0xffffffffu, l0, off);
        l1 += __shfl_xor_sync(0xffffffffu, l1, off);
    }
    if (dead) return;
    if (v0) {
        float *rec = c.ws_pre + (((int64_t)ks * c.S + members[mi0]) * c.Hkv + g) * MF;
        const int hl = r0 % G;
#pragma unroll
        for (int nd = 0; nd < ND; ++nd)
            *reinterpret_cast<float2 *>(rec + hl * D + nd * 8 + 2 * tig) = make_float2(o[nd][0], o[nd][1]);
        if (tig == 0) {
            rec[G * D + hl] = mr0;
            rec[G * D + G + hl] = l0;
        }
    }
    if (v1) {
        float *rec = c.ws_pre + (((int64_t)ks * c.S + members[mi1]) * c.Hkv + g) * MF;
        const int hl = r1 % G;
#pragma unroll
        for (int nd = 0; nd < ND; ++nd)
            *reinterpret_cast<float2 *>(rec + hl * D + nd * 8 + 2 * tig) = make_float2(o[nd][2], o[nd][3]);
        if (tig == 0) {
            rec[G * D + hl] = mr1;
            rec[G * D + G + hl] = l1;
        }
    }
}

template <int D>
inline size_t cascade_smem_bytes()
{
    return 1024 + (size_t)kPreStages * 2 * (kPreKeys / kTile) * (D / 64) * kHalfBytes + kPreStages * 8 +
           (size_t)kPreRowsCap * 4;
}

}  // namespace kvp
