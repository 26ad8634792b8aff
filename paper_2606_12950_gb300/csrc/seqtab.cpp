// seqtab.cpp -- host sequence tables: per-slot block lists and lengths over
// the shared pool, with change tracking for incremental device sync.
//
// This is the runtime's side of the paper's per-stage KV provisioning: a
// stage reserves ceil((P + L^) / bs) blocks for its predicted total length
// (Eq. 2), under-prediction grows the reservation one block at a time, a
// shared prefix is held by reference, and blocks return to the pool at the
// end of a stage or sequence (§III-C).
#include <algorithm>
#include <cstring>
#include <vector>

#include "pool_internal.h"
#include "seqtab_internal.h"

namespace {

// a table whose pool was destroyed first is detached (pool == nullptr)
bool slot_ok(const kv_seqtab *t, int s) { return t && t->pool && s >= 0 && s < t->S; }

void set_entry(kv_seqtab *t, int s, int i, int32_t v)
{
    const int64_t idx = (int64_t)s * t->max_blocks + i;
    t->table[(size_t)idx] = v;
    if (!t->pending[(size_t)idx]) {
        t->pending[(size_t)idx] = 1;
        t->changed.push_back((int32_t)idx);
    }
}

}  // namespace

void kvp_seqtab_detach(kv_seqtab *t) { t->pool = nullptr; }

extern "C" {

int kv_seqtab_create(kv_pool *pool, int layout, int max_seqs, int max_blocks, kv_seqtab **out)
{
    if (!pool || !out || layout < 0 || layout >= pool->desc.num_layouts) return KV_ERR_INVALID_ARG;
    if (max_seqs < 1 || max_blocks < 1) return KV_ERR_INVALID_ARG;
    if ((int64_t)max_seqs * max_blocks >= INT32_MAX) return KV_ERR_INVALID_ARG;
    if ((int64_t)max_blocks * pool->desc.block_size >= INT32_MAX) return KV_ERR_INVALID_ARG;
    kv_seqtab *t = new kv_seqtab();
    t->pool = pool;
    t->layout = layout;
    t->S = max_seqs;
    t->max_blocks = max_blocks;
    t->bs = pool->desc.block_size;
    t->table.assign((size_t)max_seqs * max_blocks, -1);
    t->lens.assign((size_t)max_seqs, 0);
    t->held.assign((size_t)max_seqs, 0);
    t->pending.assign((size_t)max_seqs * max_blocks, 0);
    t->full_dirty = true;
    std::memset(&t->counters, 0, sizeof t->counters);
    {
        std::lock_guard<std::mutex> g(pool->mu);
        pool->seqtabs.push_back(t);
    }
    *out = t;
    return KV_OK;
}

int kv_seq_release(kv_seqtab *t, int s)
{
    if (!slot_ok(t, s)) return KV_ERR_INVALID_ARG;
    const int h = t->held[(size_t)s];
    if (h > 0) {
        int rc = kv_free_blocks(t->pool, t->layout, h, &t->table[(size_t)s * t->max_blocks]);
        if (rc) return rc;
        for (int i = 0; i < h; ++i) set_entry(t, s, i, -1);
        t->counters.blocks_held -= h;
    }
    t->held[(size_t)s] = 0;
    t->lens[(size_t)s] = 0;
    t->counters.releases += 1;
    return KV_OK;
}

int kv_seqtab_destroy(kv_seqtab *t)
{
    if (!t) return KV_ERR_INVALID_ARG;
    int rc = KV_OK;
    if (kv_pool *pool = t->pool) {
        for (int s = 0; s < t->S; ++s)
            if (t->held[(size_t)s] > 0) {
                int r = kv_seq_release(t, s);
                if (r && !rc) rc = r;
            }
        std::lock_guard<std::mutex> g(pool->mu);
        pool->seqtabs.erase(std::remove(pool->seqtabs.begin(), pool->seqtabs.end(), t), pool->seqtabs.end());
    }
    delete t;
    return rc;
}

int kv_seq_reserve(kv_seqtab *t, int s, int64_t tokens)
{
    if (!slot_ok(t, s) || tokens < 0) return KV_ERR_INVALID_ARG;
    const int64_t need = (tokens + t->bs - 1) / t->bs;
    if (need > t->max_blocks) return KV_ERR_INVALID_ARG;
    t->counters.reserve_calls += 1;
    const int h = t->held[(size_t)s];
    if (need <= h) return KV_OK;
    const int n = (int)(need - h);
    // the new ids land in the row's free tail (all -1), then are marked changed
    int32_t *row = &t->table[(size_t)s * t->max_blocks];
    int rc = kv_alloc_blocks(t->pool, t->layout, n, row + h);
    if (rc) return rc;  // nothing written
    for (int k = 0; k < n; ++k) set_entry(t, s, h + k, row[h + k]);
    t->held[(size_t)s] = (int32_t)need;
    t->counters.blocks_held += n;
    return KV_OK;
}

int kv_seq_share_prefix(kv_seqtab *t, int dst, int src, int nblocks)
{
    if (!slot_ok(t, dst) || !slot_ok(t, src) || dst == src || nblocks < 0) return KV_ERR_INVALID_ARG;
    if (t->held[(size_t)dst] != 0 || t->lens[(size_t)dst] != 0) return KV_ERR_INVALID_ARG;
    if (t->held[(size_t)src] < nblocks || nblocks > t->max_blocks) return KV_ERR_INVALID_ARG;
    if (nblocks == 0) return KV_OK;
    const int32_t *row = &t->table[(size_t)src * t->max_blocks];
    int rc = kv_block_ref(t->pool, t->layout, nblocks, row);
    if (rc) return rc;
    for (int i = 0; i < nblocks; ++i) set_entry(t, dst, i, row[i]);
    t->held[(size_t)dst] = nblocks;
    t->counters.blocks_held += nblocks;
    return KV_OK;
}

int kv_seq_set_len(kv_seqtab *t, int s, int32_t len)
{
    if (!slot_ok(t, s) || len < 0 || (int64_t)len > (int64_t)t->held[(size_t)s] * t->bs) return KV_ERR_INVALID_ARG;
    t->lens[(size_t)s] = len;
    return KV_OK;
}

int kv_seq_advance(kv_seqtab *t, int n, const int32_t *seqs, int32_t *n_grown)
{
    if (!t || !t->pool || (seqs && n < 0)) return KV_ERR_INVALID_ARG;
    std::vector<int32_t> list;
    if (seqs) {
        list.assign(seqs, seqs + n);
        for (int32_t s : list)
            if (!slot_ok(t, s)) return KV_ERR_INVALID_ARG;
        std::vector<int32_t> sorted = list;
        std::sort(sorted.begin(), sorted.end());
        if (std::adjacent_find(sorted.begin(), sorted.end()) != sorted.end()) return KV_ERR_INVALID_ARG;
    } else {
        for (int s = 0; s < t->S; ++s)
            if (t->lens[(size_t)s] > 0) list.push_back(s);
    }
    // which slots must grow, and can they
    std::vector<int32_t> grow;
    for (int32_t s : list) {
        const int64_t len = t->lens[(size_t)s], cap = (int64_t)t->held[(size_t)s] * t->bs;
        if (len + 1 > cap) {
            if (t->held[(size_t)s] + 1 > t->max_blocks) return KV_ERR_INVALID_ARG;
            grow.push_back(s);
        }
    }
    if (!grow.empty()) {
        std::vector<int32_t> ids(grow.size());
        int rc = kv_alloc_blocks(t->pool, t->layout, (int)grow.size(), ids.data());
        if (rc) return rc;  // nothing changed
        for (size_t k = 0; k < grow.size(); ++k) {
            const int32_t s = grow[k];
            set_entry(t, s, t->held[(size_t)s], ids[k]);
            t->held[(size_t)s] += 1;
        }
        t->counters.blocks_held += (int64_t)grow.size();
        t->counters.reservation_misses += (int64_t)grow.size();
    }
    for (int32_t s : list) t->lens[(size_t)s] += 1;
    if (n_grown) *n_grown = (int32_t)grow.size();
    return KV_OK;
}

int kv_seq_trim(kv_seqtab *t, int s)
{
    if (!slot_ok(t, s)) return KV_ERR_INVALID_ARG;
    const int keep = (t->lens[(size_t)s] + t->bs - 1) / t->bs;
    const int h = t->held[(size_t)s];
    if (h <= keep) return KV_OK;
    int rc = kv_free_blocks(t->pool, t->layout, h - keep, &t->table[(size_t)s * t->max_blocks + keep]);
    if (rc) return rc;
    for (int i = keep; i < h; ++i) set_entry(t, s, i, -1);
    t->held[(size_t)s] = keep;
    t->counters.blocks_held -= h - keep;
    return KV_OK;
}

int kv_seq_replace(kv_seqtab *t, int n, const int32_t *slots, const int64_t *reserve_tokens,
                   const int32_t *lens, int32_t *status)
{
    if (!t || !t->pool || n < 0) return KV_ERR_INVALID_ARG;
    if (n == 0) return KV_OK;
    if (!slots || !reserve_tokens || !lens || !status) return KV_ERR_INVALID_ARG;
    const int64_t cap = (int64_t)t->max_blocks * t->bs;
    std::vector<uint8_t> seen((size_t)t->S, 0);
    for (int i = 0; i < n; ++i) {
        const int32_t s = slots[i];
        if (!slot_ok(t, s) || seen[(size_t)s]) return KV_ERR_INVALID_ARG;
        seen[(size_t)s] = 1;
        if (reserve_tokens[i] < 0 || reserve_tokens[i] > cap) return KV_ERR_INVALID_ARG;
        if (lens[i] < 0 || (int64_t)lens[i] > reserve_tokens[i]) return KV_ERR_INVALID_ARG;
    }
    for (int i = 0; i < n; ++i) {
        const int32_t s = slots[i];
        int rc = KV_OK;
        if (t->held[(size_t)s] > 0 || t->lens[(size_t)s] > 0) rc = kv_seq_release(t, s);
        if (rc) return rc;
        rc = kv_seq_reserve(t, s, reserve_tokens[i]);
        if (rc == KV_ERR_OUT_OF_BLOCKS) {
            status[i] = rc;  // the slot stays empty
            continue;
        }
        if (rc) return rc;
        t->lens[(size_t)s] = lens[i];
        status[i] = KV_OK;
    }
    return KV_OK;
}

int kv_seqtab_host(const kv_seqtab *t, const int32_t **table, const int32_t **ctx_lens)
{
    if (!t || !table || !ctx_lens) return KV_ERR_INVALID_ARG;
    *table = t->table.data();
    *ctx_lens = t->lens.data();
    return KV_OK;
}

int kv_seqtab_get_counters(const kv_seqtab *t, kv_seqtab_counters *out)
{
    if (!t || !out) return KV_ERR_INVALID_ARG;
    *out = t->counters;
    return KV_OK;
}

}  // extern "C"
