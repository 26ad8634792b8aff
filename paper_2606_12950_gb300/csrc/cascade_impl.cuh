// cascade_impl.cuh -- shared-prefix ("cascade") attention for sequences whose
// block tables start with the same physical blocks.
//
// Sequences that share a prefix by reference (agent stages building on one
// system prompt, §III-B / §III-C) hold identical K/V for its tokens, so the
// prefix's contribution to every sharer's decode query is one dense
// contraction per KV head: all sharers' query heads of that KV head form the
// rows, the prefix tokens the columns.  The prefix K/V is then read once per
// (row tile, key split) from L2 instead of once per sharer, and the work runs
// on the fifth-generation tensor cores as a small flash-attention forward:
//   S = Q K^T     tcgen05.mma, M = 128 query rows, N = 128 keys, fp32 in TMEM
//   softmax       one thread per row, S read from TMEM, base 2, lazy rescale
//   O += P V      tcgen05.mma, P (bf16) from TMEM, V from shared memory, O in TMEM
// with 128-key K/V tiles streamed by TMA through a 2-stage ring.  The
// softmax writes P (bf16) back over S in TMEM, and the P.V MMA reads its A
// operand from there, so P never touches shared memory.  A CTA holds two Q
// tiles that share every K/V tile: while one tile's four warps run the
// softmax, the tensor core works on the other tile.  One thread issues the
// MMAs, one warp the TMA loads, one thread owns each row.
// Each CTA leaves, per (sharer, KV head), one fp32 record (unnormalised o,
// running max m, sum l) in the same format as the decode kernel's split
// partials; the combine kernel merges prefix and suffix records, which is
// exact because the softmax over the whole context factorises over any
// partition of the keys.
#pragma once

#include "attn_impl.cuh"

namespace kvp {

constexpr int kPreRows = 128;             // query rows (sharer, head) per Q tile: the MMA's M
constexpr int kPreQTiles = 2;             // Q tiles per CTA, sharing every K/V tile
constexpr int kPreKeys = 128;             // prefix tokens per pipeline tile: S's N, P.V's K
constexpr int kPreChunk = 64;             // granularity of prefix lengths and key splits
constexpr int kPreStages = 2;
constexpr int kPreSoftWarps = 4;          // per Q tile: one thread per query row
constexpr int kPreThreads = (kPreQTiles * kPreSoftWarps + 2) * 32;  // + TMA warp + MMA warp
constexpr int kPreRowsCap = 256;          // 16-token sub-tiles resolved up front
constexpr int kMaxKeySplits = 8;
constexpr int kCascadeWords = 4080;       // most plan words (the plan kernel's parameters, then the workspace)
// TMEM per Q tile: S [0, 128) fp32, P over S's first 64 columns (bf16 pairs), O [128, 128 + d)
constexpr uint32_t kPreTmemCols = 256;

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
    int32_t overlap;      // 1: release the decode grid before the wait (it waits on the plan kernel's flags)
    // the plan in the workspace, written by the plan kernel before this grid
    // reads it: [n_groups + 1] first row tile of each group | [n_groups + 1]
    // first member index | [n_groups] prefix tokens | [n_members] member
    // sequences | [S] skip
    const int32_t *plan;
};

// members per CTA: whole query-head groups of consecutive members in each of
// its Q tiles
template <int G>
__host__ __device__ constexpr int pre_members_per_tile() { return kPreQTiles * (kPreRows / G); }

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

// shared-memory layout of the prefix kernel (offsets from a 1024-byte aligned
// base): Q [tiles][halves][128 rows][128 B] | stages x (K, V) [halves][128
// keys][128 B] | mbarriers | TMEM address | sub-tile rows
template <int D>
struct PreSmem {
    static constexpr int HALVES = D / 64;
    static constexpr uint32_t KV_HALF = kPreKeys * 128;       // 128 keys x 64 columns
    static constexpr uint32_t KV_TILE = HALVES * KV_HALF;     // K (or V) of one key tile
    static constexpr uint32_t STAGE = 2 * KV_TILE;
    static constexpr uint32_t Q_HALF = kPreRows * 128;
    static constexpr uint32_t Q_TILE = HALVES * Q_HALF;
    static constexpr uint32_t Q_OFF = 0;
    static constexpr uint32_t ST_OFF = kPreQTiles * Q_TILE;
    static constexpr uint32_t BAR_OFF = ST_OFF + kPreStages * STAGE;
    // full, empty per stage; per Q tile: s_full, p_full, o_done; fin; q_ready
    static constexpr int NBARS = 2 * kPreStages + 3 * kPreQTiles + 2;
    static constexpr uint32_t SLOT_OFF = BAR_OFF + NBARS * 8;
    static constexpr uint32_t ROWS_OFF = SLOT_OFF + 16;
    static constexpr uint32_t BYTES = ROWS_OFF + kPreRowsCap * 4;
};

template <int D, int G>
__global__ void __launch_bounds__(kPreThreads, 1)
cascade_prefix_kernel(const __grid_constant__ CUtensorMap tmap, const __grid_constant__ CascadeArgs c)
{
    using L = PreSmem<D>;
    constexpr int HALVES = L::HALVES;
    constexpr uint32_t MF = merge_floats<D, G>();
    constexpr int MQ = kPreRows / G;               // members per Q tile
    constexpr int MT = pre_members_per_tile<G>();  // members per CTA (kPreQTiles Q tiles)
    constexpr int NSUB = kPreKeys / kTile;         // 16-token sub-tiles per key tile
    constexpr int CSUB = kPreChunk / kTile;        // sub-tiles per 64-key chunk
    constexpr uint32_t O_COL = kPreKeys;           // within a Q tile's TMEM columns
    constexpr int SOFT_THREADS = kPreQTiles * kPreSoftWarps * 32;
    static_assert(O_COL + D <= kPreTmemCols, "S (with P over it) and O fit a Q tile's TMEM columns");
    extern __shared__ uint8_t smem_raw[];
    uint8_t *smem = smem_raw + ((1024u - (smem_u32(smem_raw) & 1023u)) & 1023u);
    const uint32_t sbase = smem_u32(smem);
    uint64_t *bars = reinterpret_cast<uint64_t *>(smem + L::BAR_OFF);
    uint32_t *tslot = reinterpret_cast<uint32_t *>(smem + L::SLOT_OFF);
    int32_t *rows = reinterpret_cast<int32_t *>(smem + L::ROWS_OFF);
    auto bar = [&](int i) { return smem_u32(&bars[i]); };
    constexpr int FULL = 0, EMPTY = kPreStages, QB = 2 * kPreStages, FIN = QB + 3 * kPreQTiles, Q_READY = FIN + 1;
    auto s_full = [&](int a) { return bar(QB + 3 * a); };
    auto p_full = [&](int a) { return bar(QB + 3 * a + 1); };
    auto o_done = [&](int a) { return bar(QB + 3 * a + 2); };

    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    int bid = blockIdx.x;
    const int ks = bid % c.KS;
    bid /= c.KS;
    const int g = bid % c.Hkv;
    const int tile = bid / c.Hkv;

    if (tid == 0) {
        for (int i = 0; i < kPreStages; ++i) {
            mbar_init(bar(FULL + i), 1);
            mbar_init(bar(EMPTY + i), 1);
        }
        for (int a = 0; a < kPreQTiles; ++a) {
            mbar_init(s_full(a), 1);
            mbar_init(p_full(a), kPreSoftWarps * 32);
            mbar_init(o_done(a), 1);
        }
        mbar_init(bar(FIN), 1);
        mbar_init(bar(Q_READY), SOFT_THREADS);
        fence_mbar_init();
    }
    if (warp == 0) {
        tmem_alloc(smem_u32(tslot), kPreQTiles * kPreTmemCols);
        tmem_relinquish();
    }
    if (tid == 32) prefetch_tensormap(&tmap);
    // barriers initialised and TMEM allocated: everything below may use them
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tbase = *tslot;
    bool dead = false;
    constexpr int TMA_WARP = kPreQTiles * kPreSoftWarps, MMA_WARP = TMA_WARP + 1;
    // Wait for the grid before (the plan kernel; through it the table sync
    // and the previous step's combine), then release the decode kernel that
    // follows: it runs beside this grid on the SMs this grid leaves free and
    // relies on this wait having completed in every CTA here.  When the step
    // overlaps the previous step's combine, the decode kernel waits on the
    // plan kernel's flags instead and is released first.  The plan is read
    // and the records written only after the wait: the plan kernel wrote the
    // plan, and the previous combine read the records.
    if (c.overlap) grid_launch_dependents();
    grid_dependency_wait();
    if (!c.overlap) grid_launch_dependents();

    const int32_t *tile_off = c.plan;
    const int32_t *mem_off = tile_off + c.n_groups + 1;
    const int32_t *tokens = mem_off + c.n_groups + 1;
    const int32_t *members = tokens + c.n_groups;
    // (through L2: another kernel wrote the plan)
    int grp = 0;
    while (grp + 1 < c.n_groups && __ldcg(tile_off + grp + 1) <= tile) ++grp;
    const int mo = __ldcg(mem_off + grp);
    const int m0 = mo + (tile - __ldcg(tile_off + grp)) * MT;  // this CTA's members [m0, m1)
    const int m1 = min(m0 + MT, __ldcg(mem_off + grp + 1));
    const int lead = __ldcg(members + mo);
    const int ch_all = __ldcg(tokens + grp) / kPreChunk;        // 64-key chunks of the prefix
    const int ch0 = ks * ch_all / c.KS, ch1 = (ks + 1) * ch_all / c.KS;  // non-empty: KS <= ch_all
    const int nch = ch1 - ch0;
    const int nt = (nch + 1) / 2;                                // key tiles; the last may hold one chunk
    const int nsub = nch * CSUB;
    // valid keys of key tile t: 128, or 64 for a final half tile
    auto tile_keys = [&](int t) { return min(kPreKeys, (nch - 2 * t) * kPreChunk); };

    // Q rows (member, head) of KV head g into the swizzled K-major layout the
    // MMA reads: softmax thread t fills row t % 128 of Q tile t / 128; rows
    // past the CTA's members are zero.  The MMA thread waits for q_ready.
    const int Hq = c.Hkv * G;
    const int qa_tile = tid / kPreRows, r = tid % kPreRows;  // Q tile and row of a softmax thread
    const int mrow = m0 + qa_tile * MQ + r / G;               // its member index
    const bool row_ok = tid < SOFT_THREADS && r < MQ * G && mrow < m1;
    if (tid < SOFT_THREADS) {
        const uint16_t *qrow = row_ok ? c.q + ((int64_t)__ldcg(members + mrow) * Hq + (int64_t)g * G + r % G) * D
                                      : nullptr;
        uint8_t *qdst = smem + L::Q_OFF + qa_tile * L::Q_TILE;
        uint4 qv[D / 8];
#pragma unroll
        for (int ch = 0; ch < D / 8; ++ch)
            qv[ch] = row_ok ? *reinterpret_cast<const uint4 *>(qrow + ch * 8) : make_uint4(0u, 0u, 0u, 0u);
#pragma unroll
        for (int ch = 0; ch < D / 8; ++ch)
            *reinterpret_cast<uint4 *>(qdst + (ch / 8) * L::Q_HALF + swz(r, ch % 8)) = qv[ch];
        fence_proxy_async_smem();  // Q (generic stores) is read by the tensor cores
        mbar_arrive(bar(Q_READY));
    }

    if (warp == TMA_WARP) {
        // ---- TMA producer warp: resolves the pool rows of the CTA's key range
        // from the block table, then streams K and V of key tile t into stage
        // t % stages, one box per lane (one issuing thread per SM cannot keep
        // the loads flowing) ----
        for (int i = lane; i < min(nsub, kPreRowsCap); i += 32) rows[i] = pre_sub_row(c, lead, g, ch0 * CSUB + i);
        __syncwarp();
        const uint64_t pol = l2_policy_evict_normal();  // the prefix is re-read by every row tile
        constexpr int NBOX = NSUB * HALVES;               // boxes of K (and of V) per full key tile
        static_assert(2 * NBOX <= 32, "one box per lane");
        for (int t = 0; t < nt; ++t) {
            const int st = t % kPreStages;
            if (t >= kPreStages) wait_phase(bar(EMPTY + st), (uint32_t)(t / kPreStages - 1) & 1u, c.err, dead);
            const int vsub = tile_keys(t) / kTile;        // sub-tiles loaded this tile
            const uint32_t kdst = sbase + L::ST_OFF + st * L::STAGE, vdst = kdst + L::KV_TILE;
            const int box = lane % NBOX, j = box / HALVES, h = box % HALVES;
            const bool mine = lane < 2 * NBOX && j < vsub;
            int32_t y = 0;
            bool ok = true;
            if (mine) {
                const int32_t q = t * NSUB + j;
                y = q < kPreRowsCap ? rows[q] : pre_sub_row(c, lead, g, ch0 * CSUB + q);
                ok = y >= 0;
            }
            ok = __all_sync(0xffffffffu, ok);
            if (!ok) {
                if (lane == 0) {
                    report(c.err, KV_ERR_DEVICE_BOUNDS);
                    mbar_arrive(bar(FULL + st));  // complete the phase without data
                }
                __syncwarp();
                continue;
            }
            if (lane == 0) mbar_arrive_expect_tx(bar(FULL + st), 2u * vsub * HALVES * (kTile * 128));
            __syncwarp();
            if (mine) {
                const uint32_t off = h * L::KV_HALF + j * (kTile * 128);
                if (lane < NBOX)
                    tma_load_2d(kdst + off, &tmap, h * 64, y, bar(FULL + st), pol);
                else
                    tma_load_2d(vdst + off, &tmap, h * 64, y + c.Hkv * c.bs, bar(FULL + st), pol);
            }
            __syncwarp();
        }
        // drain: the last stages' loads have landed (already waited on by the
        // MMA thread unless a wait ran out)
        if (lane == 0)
            for (int t = max(0, nt - kPreStages); t < nt; ++t)
                wait_phase(bar(FULL + t % kPreStages), (uint32_t)(t / kPreStages) & 1u, c.err, dead);
    } else if (warp == MMA_WARP && lane == 0) {
        // ---- MMA issuer.  Per Q tile a and key tile t: S_a = Q_a K_t^T into
        // TMEM, then, once the tile's warps have written P (bf16) over S,
        // O_a += P V_t with P read from TMEM.  The tensor pipe runs one
        // thread's MMAs in issue order, so S_a(t+1), issued after
        // P.V_a(t), overwrites P only after that MMA has read it.  Order:
        // S_0(0) S_1(0) | PV_0(t) S_0(t+1) PV_1(t) S_1(t+1) | ... ----
        constexpr uint32_t ID_S = idesc_bf16_f32(kPreRows, kPreKeys, 0, 0);
        constexpr uint32_t ID_S_HALF = idesc_bf16_f32(kPreRows, kPreChunk, 0, 0);
        constexpr uint32_t ID_O = idesc_bf16_f32(kPreRows, D, 0, 1);
        auto issue_s = [&](int a, int t) {
            const uint32_t ka = sbase + L::ST_OFF + (t % kPreStages) * L::STAGE;
            const uint32_t qa = sbase + L::Q_OFF + a * L::Q_TILE;
            const uint32_t id = tile_keys(t) == kPreKeys ? ID_S : ID_S_HALF;
#pragma unroll
            for (int kk = 0; kk < D / 16; ++kk)
                umma_bf16(tbase + a * kPreTmemCols, smem_desc_sw128(qa + (kk / 4) * L::Q_HALF + (kk % 4) * 32, 16, 1024),
                          smem_desc_sw128(ka + (kk / 4) * L::KV_HALF + (kk % 4) * 32, 16, 1024), id, kk > 0);
            umma_commit(s_full(a));
        };
        auto issue_pv = [&](int a, int t) {
            const uint32_t va = sbase + L::ST_OFF + (t % kPreStages) * L::STAGE + L::KV_TILE;
            const int ksteps = tile_keys(t) / 16;
            for (int kk = 0; kk < ksteps; ++kk)
                umma_bf16_tmem_a(tbase + a * kPreTmemCols + O_COL, tbase + a * kPreTmemCols + kk * 8,
                                 smem_desc_sw128(va + kk * (16 * 128), L::KV_HALF, 1024), ID_O, t > 0 || kk > 0);
            umma_commit(o_done(a));
        };
        wait_phase(bar(Q_READY), 0u, c.err, dead);
        wait_phase(bar(FULL + 0), 0u, c.err, dead);
        tc_fence_after();
        for (int a = 0; a < kPreQTiles; ++a) issue_s(a, 0);
        for (int t = 0; t < nt; ++t) {
            const bool next = t + 1 < nt;
            for (int a = 0; a < kPreQTiles; ++a) {
                wait_phase(p_full(a), (uint32_t)t & 1u, c.err, dead);
                tc_fence_after();
                issue_pv(a, t);
                if (a == kPreQTiles - 1) umma_commit(bar(EMPTY + t % kPreStages));
                if (next) {
                    if (a == 0) wait_phase(bar(FULL + (t + 1) % kPreStages), (uint32_t)((t + 1) / kPreStages) & 1u,
                                           c.err, dead);
                    tc_fence_after();
                    issue_s(a, t + 1);
                }
            }
        }
        // every MMA of this thread has completed before TMEM is released
        umma_commit(bar(FIN));
        wait_phase(bar(FIN), 0u, c.err, dead);
    } else if (tid < SOFT_THREADS) {
        // ---- softmax: thread tid owns row r of Q tile qa_tile (TMEM lane r) ----
        const int a = qa_tile;
        const uint32_t trow = tbase + a * kPreTmemCols + ((uint32_t)((warp % 4) * 32) << 16);
        const float scale = c.qk_scale;
        float m_run = -INFINITY, l_run = 0.f;
        for (int t = 0; t < nt; ++t) {
            const int nk = tile_keys(t);  // 128 or 64
            // S_a(t) complete: so is every earlier MMA of the tile, in
            // particular P.V_a(t-1), so O is stable and P's columns are free
            wait_phase(s_full(a), (uint32_t)t & 1u, c.err, dead);
            tc_fence_after();
            // One pass over the tile, 64 keys (one chunk) at a time: p =
            // 2^(s * scale - m_ref) as bf16 pairs written over the first
            // columns of S (the A operand of P.V; chunk cp's 32 words land on
            // columns 32cp .. 32cp + 31, which hold scores already read).
            // m_ref is the running max, raised (lazy rescale) only when a
            // chunk exceeds it by more than 2^8: then O, l, this tile's sum
            // and the P words already written for it are scaled by
            // 2^(m_old - m_new) first, so every stored p stays <= 2^8 and
            // o, l and P share one reference max.
            float rs = 0.f;
#pragma unroll
            for (int cp = 0; cp < kPreKeys / 64; ++cp) {
                if (cp * 64 >= nk) break;
                uint32_t v[2][32];
                tmem_ld32(trow + cp * 64, v[0]);
                tmem_ld32(trow + cp * 64 + 32, v[1]);
                tmem_wait_ld();
                float mx[4] = {-INFINITY, -INFINITY, -INFINITY, -INFINITY};
#pragma unroll
                for (int i = 0; i < 64; ++i) mx[i & 3] = fmaxf(mx[i & 3], __uint_as_float(v[i >> 5][i & 31]));
                const float cmax = fmaxf(fmaxf(mx[0], mx[1]), fmaxf(mx[2], mx[3])) * scale;
                if (cmax > m_run + 8.f) {
                    const float al = fast_exp2(m_run - cmax);  // 0 when nothing came before
                    l_run *= al;
                    rs *= al;
                    if (t >= 1) {  // O holds earlier tiles
                        uint32_t o[32];
#pragma unroll
                        for (int cb = 0; cb < D / 32; ++cb) {
                            tmem_ld32(trow + O_COL + cb * 32, o);
                            tmem_wait_ld();
#pragma unroll
                            for (int i = 0; i < 32; ++i) o[i] = __float_as_uint(__uint_as_float(o[i]) * al);
                            tmem_st32(trow + O_COL + cb * 32, o);
                        }
                    }
                    for (int cq = 0; cq < cp; ++cq) {  // this tile's earlier P words
                        uint32_t w[32];
                        tmem_ld32(trow + cq * 32, w);
                        tmem_wait_ld();
#pragma unroll
                        for (int i = 0; i < 32; ++i)
                            w[i] = pack_bf16(__uint_as_float(w[i] << 16) * al, __uint_as_float(w[i] & 0xFFFF0000u) * al);
                        tmem_st32(trow + cq * 32, w);
                    }
                    m_run = cmax;
                }
                uint32_t w[32];
                float r4[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
                for (int i = 0; i < 64; i += 2) {
                    const float p0 = fast_exp2(fmaf(__uint_as_float(v[i >> 5][i & 31]), scale, -m_run));
                    const float p1 = fast_exp2(fmaf(__uint_as_float(v[i >> 5][(i + 1) & 31]), scale, -m_run));
                    r4[(i >> 1) & 3] += p0 + p1;
                    w[i / 2] = pack_bf16(p0, p1);
                }
                rs += (r4[0] + r4[1]) + (r4[2] + r4[3]);
                tmem_st32(trow + cp * 32, w);
            }
            l_run += rs;
            tmem_wait_st();
            tc_fence_before();
            mbar_arrive(p_full(a));
        }
        // ---- this CTA's record per (sharer, KV head) ----
        wait_phase(o_done(a), (uint32_t)(nt - 1) & 1u, c.err, dead);
        tc_fence_after();
        float *rec = row_ok ? c.ws_pre + (((int64_t)ks * c.S + __ldcg(members + mrow)) * c.Hkv + g) * MF : nullptr;
        const int hl = r % G;
        uint32_t v[32];
#pragma unroll
        for (int cb = 0; cb < D / 32; ++cb) {
            tmem_ld32(trow + O_COL + cb * 32, v);
            tmem_wait_ld();
            if (row_ok && !dead)
#pragma unroll
                for (int i = 0; i < 32; i += 4)
                    *reinterpret_cast<float4 *>(rec + hl * D + cb * 32 + i) =
                        make_float4(__uint_as_float(v[i]), __uint_as_float(v[i + 1]), __uint_as_float(v[i + 2]),
                                    __uint_as_float(v[i + 3]));
        }
        if (row_ok && !dead) {
            rec[G * D + hl] = m_run;
            rec[G * D + G + hl] = l_run;
        }
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    if (warp == 0) tmem_dealloc(tbase, kPreQTiles * kPreTmemCols);
}

template <int D>
inline size_t cascade_smem_bytes()
{
    return 1024 + (size_t)PreSmem<D>::BYTES;
}

}  // namespace kvp
