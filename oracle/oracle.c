/*
 * oracle.c -- plain, slow, fp64 CPU oracle for paged decode attention and
 * KV append.  TEST INFRASTRUCTURE ONLY: the library's product path never
 * links, loads or calls this file; only the tests, the smoke check and the
 * benchmark's CPU-baseline leg do.
 *
 * What it computes (the decode phase of §II "LLM inference cost model": one
 * new token per sequence attends over the whole cached context, whose KV grows
 * linearly with P+L; the cache is block-paged as the PagedAttention engine the
 * paper builds on (§II, §IV-A) and as the shared KV pool of §III-C):
 *
 *   For sequence s with post-append length n, query head h, KV head
 *   g = floor(h / G) with G = Hq / Hkv, and positions j = 0 .. n-1 resolved
 *   through the block table (blk = table[s][j / bs], off = j % bs):
 *
 *     x_j  = scale * sum_c q[s][h][c] * K(blk, g, off, c)
 *     p_j  = exp(x_j - max_i x_i) / sum_i exp(x_i - max_i x_i)
 *     o[c] = sum_j p_j * V(blk, g, off, c)
 *
 *   Append writes the bf16 bits of k_new[s][g][:] and v_new[s][g][:] into the
 *   slot of position n-1; every other pool element is untouched.
 *
 * Pool layout: element units are bf16 (uint16).  Block id b starts at element
 * b * page_elems.  Inside a block of a layout with Hkv heads, block size bs
 * and head dim d the order is [K|V][Hkv][bs][d]:
 *   K(b, g, off, c) = pool[b*page_elems + ((0*Hkv + g)*bs + off)*d + c]
 *   V(b, g, off, c) = pool[b*page_elems + ((1*Hkv + g)*bs + off)*d + c]
 *
 * A sequence with n = 0 has no defined softmax; the oracle returns zeros for
 * it (the library's stated convention).
 *
 * Everything is accumulated in fp64 in natural position order; exp is the C
 * library's.  The functions return 0, or -1 if an index leaves the pool or
 * the table (nothing is written in that case for attention; append stops at
 * the first bad row).
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

static double bf16_to_double(uint16_t bits)
{
    uint32_t u = ((uint32_t)bits) << 16;
    float f;
    memcpy(&f, &u, sizeof f);
    return (double)f;
}

/* element offset of K (which = 0) or V (which = 1) for (block, head, off, c) */
static int64_t kv_elem(int64_t block, int64_t page_elems, int which, int g, int off,
                       int c, int Hkv, int bs, int d)
{
    return block * page_elems + (((int64_t)which * Hkv + g) * bs + off) * d + c;
}

/* check that a table entry names a whole block inside the pool */
static int block_ok(int64_t block, int64_t page_elems, int64_t n_pages, int Hkv, int bs,
                    int d)
{
    int64_t block_elems = 2LL * Hkv * bs * d;
    if (block < 0) return 0;
    return block * page_elems + block_elems <= n_pages * page_elems;
}

int oracle_append(uint16_t *pool, int64_t n_pages, int64_t page_elems, int bs, int Hkv,
                  int d, const uint16_t *k_new, const uint16_t *v_new,
                  const int32_t *table, const int32_t *ctx_lens, int max_blocks, int S)
{
    for (int s = 0; s < S; ++s) {
        int n = ctx_lens[s];
        if (n <= 0) continue; /* nothing to append into */
        int pos = n - 1;
        int lb = pos / bs;
        if (lb >= max_blocks) return -1;
        int64_t blk = table[(int64_t)s * max_blocks + lb];
        if (!block_ok(blk, page_elems, n_pages, Hkv, bs, d)) return -1;
        int off = pos % bs;
        for (int g = 0; g < Hkv; ++g) {
            for (int c = 0; c < d; ++c) {
                pool[kv_elem(blk, page_elems, 0, g, off, c, Hkv, bs, d)] =
                    k_new[((int64_t)s * Hkv + g) * d + c];
                pool[kv_elem(blk, page_elems, 1, g, off, c, Hkv, bs, d)] =
                    v_new[((int64_t)s * Hkv + g) * d + c];
            }
        }
    }
    return 0;
}

/* Attention for one (s, h); writes d doubles to o.  Scratch x holds n scores. */
static int attend_one(const uint16_t *pool, int64_t n_pages, int64_t page_elems, int bs,
                      int Hkv, int d, const uint16_t *qrow, const int32_t *trow, int n,
                      int max_blocks, int g, double scale, double *x, double *o)
{
    for (int c = 0; c < d; ++c) o[c] = 0.0;
    if (n <= 0) return 0;
    if ((n + bs - 1) / bs > max_blocks) return -1;
    /* scores */
    for (int j = 0; j < n; ++j) {
        int64_t blk = trow[j / bs];
        if (!block_ok(blk, page_elems, n_pages, Hkv, bs, d)) return -1;
        int off = j % bs;
        double acc = 0.0;
        for (int c = 0; c < d; ++c)
            acc += bf16_to_double(qrow[c]) *
                   bf16_to_double(pool[kv_elem(blk, page_elems, 0, g, off, c, Hkv, bs, d)]);
        x[j] = scale * acc;
    }
    /* softmax */
    double m = x[0];
    for (int j = 1; j < n; ++j)
        if (x[j] > m) m = x[j];
    double denom = 0.0;
    for (int j = 0; j < n; ++j) {
        x[j] = exp(x[j] - m);
        denom += x[j];
    }
    /* weighted sum of values */
    for (int j = 0; j < n; ++j) {
        int64_t blk = trow[j / bs];
        int off = j % bs;
        double p = x[j] / denom;
        for (int c = 0; c < d; ++c)
            o[c] += p * bf16_to_double(pool[kv_elem(blk, page_elems, 1, g, off, c, Hkv, bs, d)]);
    }
    return 0;
}

/*
 * out: fp64 [S][Hq][d].  If seq_ids is non-NULL only the n_ids listed
 * sequences are computed (their rows of out are written, others untouched).
 */
int oracle_paged_attention(const uint16_t *pool, int64_t n_pages, int64_t page_elems,
                           int bs, int Hkv, int d, const uint16_t *q,
                           const int32_t *table, const int32_t *ctx_lens, int max_blocks,
                           int S, int Hq, double scale, const int32_t *seq_ids, int n_ids,
                           double *out)
{
    if (Hkv <= 0 || Hq % Hkv != 0) return -1;
    int G = Hq / Hkv;
    int count = seq_ids ? n_ids : S;
    int nmax = 0;
    for (int i = 0; i < count; ++i) {
        int s = seq_ids ? seq_ids[i] : i;
        if (s < 0 || s >= S) return -1;
        if (ctx_lens[s] > nmax) nmax = ctx_lens[s];
    }
    double *x = (double *)malloc(sizeof(double) * (size_t)(nmax > 0 ? nmax : 1));
    if (!x) return -1;
    int rc = 0;
    for (int i = 0; i < count && rc == 0; ++i) {
        int s = seq_ids ? seq_ids[i] : i;
        for (int h = 0; h < Hq && rc == 0; ++h) {
            rc = attend_one(pool, n_pages, page_elems, bs, Hkv, d,
                            q + ((int64_t)s * Hq + h) * d, table + (int64_t)s * max_blocks,
                            ctx_lens[s], max_blocks, h / G, scale, x,
                            out + ((int64_t)s * Hq + h) * d);
        }
    }
    free(x);
    return rc;
}

/*
 * Dense attention on gathered arrays, for pinning the paged version:
 * k, v are fp64 [Hkv][n][d], q fp64 [Hq][d], out fp64 [Hq][d].
 */
int oracle_dense_attention(const double *q, const double *k, const double *v, int n,
                           int Hq, int Hkv, int d, double scale, double *out)
{
    if (Hkv <= 0 || Hq % Hkv != 0) return -1;
    int G = Hq / Hkv;
    double *x = (double *)malloc(sizeof(double) * (size_t)(n > 0 ? n : 1));
    if (!x) return -1;
    for (int h = 0; h < Hq; ++h) {
        int g = h / G;
        double *o = out + (int64_t)h * d;
        for (int c = 0; c < d; ++c) o[c] = 0.0;
        if (n <= 0) continue;
        double m = -INFINITY;
        for (int j = 0; j < n; ++j) {
            double acc = 0.0;
            for (int c = 0; c < d; ++c)
                acc += q[(int64_t)h * d + c] * k[((int64_t)g * n + j) * d + c];
            x[j] = scale * acc;
            if (x[j] > m) m = x[j];
        }
        double denom = 0.0;
        for (int j = 0; j < n; ++j) {
            x[j] = exp(x[j] - m);
            denom += x[j];
        }
        for (int j = 0; j < n; ++j)
            for (int c = 0; c < d; ++c)
                o[c] += x[j] / denom * v[((int64_t)g * n + j) * d + c];
    }
    free(x);
    return 0;
}

/*
 * Split-K form of the same attention (what a split decode computes): the
 * positions of one (s, h) are cut into consecutive splits of split_len
 * tokens.  Split i yields m_i = max of its scores, l_i = sum exp(x - m_i),
 * u_i[c] = sum exp(x - m_i) v[c].  The combine takes M = max_i m_i and
 * o = sum_i e^{m_i - M} u_i / sum_i e^{m_i - M} l_i.  In exact arithmetic this
 * equals the unsplit softmax for every split_len.
 *
 * out: fp64 [S][Hq][d].
 */
static int split_partial(const uint16_t *pool, int64_t n_pages, int64_t page_elems, int bs,
                         int Hkv, int d, const uint16_t *qrow, const int32_t *trow, int g,
                         double scale, int start, int end, double *m_out, double *l_out,
                         double *u)
{
    double mi = -INFINITY;
    for (int j = start; j < end; ++j) {
        int64_t blk = trow[j / bs];
        if (!block_ok(blk, page_elems, n_pages, Hkv, bs, d)) return -1;
        double acc = 0.0;
        for (int c = 0; c < d; ++c)
            acc += bf16_to_double(qrow[c]) *
                   bf16_to_double(pool[kv_elem(blk, page_elems, 0, g, j % bs, c, Hkv, bs, d)]);
        if (scale * acc > mi) mi = scale * acc;
    }
    double li = 0.0;
    for (int c = 0; c < d; ++c) u[c] = 0.0;
    for (int j = start; j < end; ++j) {
        int64_t blk = trow[j / bs];
        double acc = 0.0;
        for (int c = 0; c < d; ++c)
            acc += bf16_to_double(qrow[c]) *
                   bf16_to_double(pool[kv_elem(blk, page_elems, 0, g, j % bs, c, Hkv, bs, d)]);
        double e = exp(scale * acc - mi);
        li += e;
        for (int c = 0; c < d; ++c)
            u[c] += e * bf16_to_double(pool[kv_elem(blk, page_elems, 1, g, j % bs, c, Hkv, bs, d)]);
    }
    *m_out = mi;
    *l_out = li;
    return 0;
}

int oracle_split_attention(const uint16_t *pool, int64_t n_pages, int64_t page_elems,
                           int bs, int Hkv, int d, const uint16_t *q,
                           const int32_t *table, const int32_t *ctx_lens, int max_blocks,
                           int S, int Hq, double scale, int split_len, double *out)
{
    if (Hkv <= 0 || Hq % Hkv != 0 || split_len <= 0) return -1;
    int G = Hq / Hkv;
    int nmax = 0;
    for (int s = 0; s < S; ++s)
        if (ctx_lens[s] > nmax) nmax = ctx_lens[s];
    int max_splits = (nmax + split_len - 1) / split_len;
    if (max_splits < 1) max_splits = 1;
    double *m = (double *)malloc(sizeof(double) * (size_t)max_splits);
    double *l = (double *)malloc(sizeof(double) * (size_t)max_splits);
    double *u = (double *)malloc(sizeof(double) * (size_t)max_splits * (size_t)d);
    int rc = (m && l && u) ? 0 : -1;
    for (int s = 0; s < S && rc == 0; ++s) {
        int n = ctx_lens[s];
        if ((n + bs - 1) / bs > max_blocks) { rc = -1; break; }
        const int32_t *trow = table + (int64_t)s * max_blocks;
        int ns = (n + split_len - 1) / split_len;
        for (int h = 0; h < Hq && rc == 0; ++h) {
            const uint16_t *qrow = q + ((int64_t)s * Hq + h) * d;
            double *o = out + ((int64_t)s * Hq + h) * d;
            for (int c = 0; c < d; ++c) o[c] = 0.0;
            if (n <= 0) continue;
            /* partials of every split */
            for (int i = 0; i < ns && rc == 0; ++i) {
                int start = i * split_len;
                int end = start + split_len < n ? start + split_len : n;
                rc = split_partial(pool, n_pages, page_elems, bs, Hkv, d, qrow, trow, h / G,
                                   scale, start, end, &m[i], &l[i], u + (int64_t)i * d);
            }
            if (rc) break;
            /* combine */
            double M = m[0];
            for (int i = 1; i < ns; ++i)
                if (m[i] > M) M = m[i];
            double denom = 0.0;
            for (int i = 0; i < ns; ++i) {
                double w = exp(m[i] - M);
                denom += w * l[i];
                for (int c = 0; c < d; ++c) o[c] += w * u[(int64_t)i * d + c];
            }
            for (int c = 0; c < d; ++c) o[c] /= denom;
        }
    }
    free(m);
    free(l);
    free(u);
    return rc;
}
