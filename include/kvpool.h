/*
 * kvpool.h -- C ABI of libkvpool: one block-paged bf16 KV pool in HBM shared
 * by many sequences (and several model layouts), the per-step append of each
 * sequence's new K/V row, and batched paged decode attention over the pool.
 *
 * What the paper fixes and what it leaves to us
 * ---------------------------------------------
 * The paper (Maestro, a workload-aware scheduler for multi-agent LLM serving)
 * treats this path as the engine under its runtime:
 *   - KV footprint grows linearly with prompt + output length (§II, "KV cache
 *     memory pressure"); per stage the runtime reserves alpha(M) * (P + L^)
 *     of it (Eq. 2).
 *   - One GPU's KV lives in a single shared pool whose pages are handed out
 *     on demand to the stages of co-located models; when physical memory runs
 *     out the stage is rejected, not crashed (§III-C, "Spatial multiplexing
 *     with virtual-memory KV cache"; explicit accounting M_kv + M_res <= M_total).
 *   - The serving engine pages the cache into fixed-size blocks reached
 *     through a per-sequence block table (PagedAttention, §II and §IV-A).
 *   - Decode dominates latency for long outputs (§II, "LLM inference cost
 *     model"): every step, every live sequence attends with one new query over
 *     its whole cached context.
 * The paper gives no API, no layout and no kernel; those are this library's.
 *
 * Conventions (all entry points)
 * ------------------------------
 *   - Every function returns an int: KV_OK (0) or a negative kv_status.
 *   - The caller owns ALL device memory (pool, tables, lengths, q, out,
 *     workspace, error word) and all streams; pointers are plain device
 *     addresses and cudaStream_t handles passed as void*.  The library owns only
 *     host-side metadata (free lists, refcounts).
 *   - Launches are asynchronous on the given stream (NULL = legacy default
 *     stream).  Argument errors are detected on the host before anything is
 *     launched and leave every buffer untouched.
 *   - bf16 tensors are IEEE bfloat16 bit patterns (uint16), row-major and
 *     contiguous.  Outputs are rounded fp32 -> bf16 to nearest-even.
 *   - Out-of-range indices found on the device (a table entry outside the
 *     pool, a context length beyond the table) never fault: the access is
 *     skipped, the error word is set to KV_ERR_DEVICE_BOUNDS, and the results
 *     of the affected sequence are unspecified.  Read it with
 *     kv_pool_get_error().
 *
 * Pool layout
 * -----------
 * The pool is cut into pages of page_bytes.  A block of layout L (Hkv KV
 * heads, head dim d, block size bs tokens) occupies block_bytes(L) =
 * 2 * Hkv * bs * d * 2 bytes = k_L consecutive pages, and is named by the id
 * of its first page.  Block id b starts at byte b * page_bytes and holds
 *     [K|V][Hkv][bs][d]  (bf16),
 * so the K (or V) tile of one KV head is one contiguous bs*d*2-byte run.
 * Token j of a sequence lives in block table[s][j / bs] at offset j % bs.
 */
#ifndef KVPOOL_H
#define KVPOOL_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum kv_status {
    KV_OK = 0,
    KV_ERR_INVALID_ARG = -1,   /* bad pointer, size, id or layout; nothing launched */
    KV_ERR_OUT_OF_BLOCKS = -2, /* allocation cannot be met; nothing allocated */
    KV_ERR_CUDA = -3,          /* a CUDA runtime call failed */
    KV_ERR_DEVICE_BOUNDS = -4, /* (error word) a device-side index check failed */
    KV_ERR_UNSUPPORTED = -5,   /* shape not built into this library (d, G) */
    KV_ERR_WORKSPACE = -6,     /* workspace missing or smaller than kv_workspace_bytes() */
    KV_ERR_DEVICE_TIMEOUT = -7 /* (error word) a bounded device wait gave up */
} kv_status;

#define KV_MAX_LAYOUTS 4

/* Geometry of one model's layer KV in the pool. */
typedef struct kv_layout {
    int32_t num_kv_heads; /* Hkv >= 1 */
    int32_t head_dim;     /* d: 64 or 128 */
} kv_layout;

typedef struct kv_pool_desc {
    void *device_base;     /* caller-owned device buffer, 256-byte aligned */
    uint64_t pool_bytes;   /* its size; pages = pool_bytes / page_bytes */
    int32_t block_size;    /* bs: tokens per block, 1..256, same for all layouts */
    int32_t num_layouts;   /* 1..KV_MAX_LAYOUTS */
    kv_layout layouts[KV_MAX_LAYOUTS];
    uint64_t page_bytes;   /* 0 = smallest layout block; every layout's block
                              bytes must be a multiple of it, and it a multiple of 256 */
    int32_t *device_error; /* caller-owned device int32, zero-initialised */
    uint64_t shuffle_seed; /* 0: free list hands out ascending ids; otherwise the
                              initial free order is a seeded permutation
                              (splitmix64 Fisher-Yates) to scatter placement */
} kv_pool_desc;

typedef struct kv_pool kv_pool;

typedef struct kv_stats {
    int64_t pages_total;
    int64_t pages_unassigned;                /* whole free superpages */
    int64_t blocks_used[KV_MAX_LAYOUTS];     /* blocks with refcount > 0 */
    int64_t blocks_cached[KV_MAX_LAYOUTS];   /* free blocks held by the layout */
    int64_t blocks_capacity[KV_MAX_LAYOUTS]; /* used + cached + unassigned/k */
    uint64_t bytes_used;                     /* sum of used blocks' bytes */
    uint64_t bytes_total;                    /* pages_total * page_bytes */
    uint64_t bytes_mapped;                   /* physically backed bytes (VMM pool); bytes_total otherwise */
    int64_t attn_calls_overlapped;           /* attention calls that started while the previous
                                                call's combine finished (kv_set_attn_step_overlap) */
} kv_stats;

/* ---------------------------------------------------------------- pool --- */

/*
 * Create the host-side manager of a caller-owned device pool (§III-C: one
 * shared KV pool per GPU, pages handed out per stage).  Allocation is a slab
 * scheme: pages are grouped into superpages of K = max_L k_L pages; a layout
 * takes a whole free superpage when its own free list is empty and cuts it
 * into K / k_L blocks.  Freed blocks go back to their layout's LIFO free list.
 * Also queries the current device (SM count) for launch sizing.
 * Errors: KV_ERR_INVALID_ARG (null/misaligned pointers, bad geometry, pool
 * smaller than one superpage), KV_ERR_CUDA.
 */
int kv_pool_create(const kv_pool_desc *desc, kv_pool **out_pool);

/* Release host metadata.  The device buffer of a fixed pool is the caller's;
 * a VMM pool's mappings and reserved range are released (after a device
 * synchronize when the library's CUDA backend owns them). */
int kv_pool_destroy(kv_pool *pool);

/*
 * VMM-backed elastic pool (§III-C, spatial multiplexing with a virtual-memory
 * KV cache).  The pool's pool_bytes are a reserved virtual range that may
 * exceed the physical memory the KV may use (overcommitment, Table 5); it is
 * cut into chunks of chunk_bytes (a multiple of the superpage, so superpages
 * never straddle chunks) that are physically mapped when kv_alloc_blocks
 * needs their superpages, and unmapped by kv_pool_trim.  kv_alloc_blocks maps
 * first and allocates after, all-or-nothing: a chunk that cannot be mapped
 * (device memory exhausted, physical_limit or the shared budget reached)
 * rejects the request with KV_ERR_OUT_OF_BLOCKS and allocates nothing.
 *
 * Backends:
 *   map_fn == NULL: CUDA virtual memory management on `device`.  The library
 *     reserves the range (desc->device_base must be NULL; read it back with
 *     kv_pool_get_base), chunk_bytes 0 = the allocation granularity (else a
 *     multiple of it), and backs every unmapped chunk with one shared guard
 *     allocation, so a device table entry naming an unallocated block reads
 *     zeros or stale data instead of faulting.
 *   map_fn != NULL: the caller's backing over its own range desc->device_base
 *     (e.g. a framework's allocator, or a host fake in tests): the library
 *     calls map_fn(ctx, offset, bytes) / unmap_fn(ctx, offset, bytes) per
 *     chunk (0 = success) and chunk_bytes must be given.
 * The pool covers whole chunks (pool_bytes is rounded down).  Block tables
 * uploaded with kv_block_table_upload may name only blocks in mapped chunks.
 * Errors: KV_ERR_INVALID_ARG, KV_ERR_CUDA (reservation or guard mapping).
 */
typedef struct kv_budget kv_budget;

typedef struct kv_vmm_desc {
    uint64_t chunk_bytes;     /* mapping unit; 0 = granularity (CUDA backend only) */
    uint64_t physical_limit;  /* at most this many bytes mapped in this pool; 0 = no limit */
    kv_budget *budget;        /* optional limit shared by several pools (mapped bytes of all of them) */
    int32_t device;           /* CUDA device ordinal (CUDA backend) */
    int32_t reserved;
    int (*map_fn)(void *ctx, uint64_t offset, uint64_t bytes);
    int (*unmap_fn)(void *ctx, uint64_t offset, uint64_t bytes);
    void *ctx;
} kv_vmm_desc;

int kv_pool_create_vmm(const kv_pool_desc *desc, const kv_vmm_desc *vmm, kv_pool **out_pool);

/* Device address of the pool's first byte (the reserved range of a VMM pool). */
int kv_pool_get_base(const kv_pool *pool, void **base);

/*
 * Give memory back: superpages whose blocks are all free return from their
 * layout's free list to the shared list (so other layouts can use them), and
 * a VMM pool unmaps every chunk whose superpages are all free, adding the
 * bytes to *released_bytes (may be NULL).  The CUDA backend synchronises the
 * device before unmapping (kernels in flight may still read freed blocks).
 */
int kv_pool_trim(kv_pool *pool, uint64_t *released_bytes);

/* A physical-memory budget shared by VMM pools (e.g. M_total - M_res of the
 * node, §III-C).  Destroy it after every pool that uses it. */
int kv_budget_create(uint64_t limit_bytes, kv_budget **out);
int kv_budget_destroy(kv_budget *budget);
int kv_budget_used(const kv_budget *budget, uint64_t *used_bytes);

/*
 * Reserve n blocks of layout `layout` (Eq. 2's per-stage reservation is n =
 * ceil((P + L^) / bs) blocks; the caller decides n).  Writes n block ids
 * (refcount 1) to the host array out_ids.  All-or-nothing: on
 * KV_ERR_OUT_OF_BLOCKS nothing is allocated (§III-C: a stage whose memory
 * cannot be mapped is rejected).
 */
int kv_alloc_blocks(kv_pool *pool, int layout, int n, int32_t *out_ids);

/*
 * Drop one reference to each of n blocks (host array).  A block whose count
 * reaches zero returns to its layout's free list.  Validated before anything
 * changes: every id must be a live block of `layout` holding at least as many
 * references as it appears in ids, else KV_ERR_INVALID_ARG.
 */
int kv_free_blocks(kv_pool *pool, int layout, int n, const int32_t *ids);

/*
 * Add one reference to each of n live blocks of `layout` (a prefix shared by
 * reference by several block tables).  Validated first; KV_ERR_INVALID_ARG.
 */
int kv_block_ref(kv_pool *pool, int layout, int n, const int32_t *ids);

/* Refcount of a block id (0 = free), or KV_ERR_INVALID_ARG for a bad id. */
int kv_block_refcount(const kv_pool *pool, int32_t id, int32_t *out_count);

/* Counters of the pool (host only). */
int kv_pool_stats(const kv_pool *pool, kv_stats *out);

/*
 * Asynchronously copy the device error word into *host_code (host memory; use
 * pinned memory for true asynchrony) and reset it to zero, on `stream`.  The
 * value is valid after the stream reaches this point (e.g. after
 * cudaStreamSynchronize).  0 means no device-side error since the last call.
 */
int kv_pool_get_error(kv_pool *pool, void *stream, int32_t *host_code);

/* ------------------------------------------------------- block tables --- */

/*
 * Copy a block table and context lengths from host to device on `stream`:
 * host_table int32 [S][max_blocks] -> dev_table, host_ctx_lens int32 [S] ->
 * dev_ctx_lens.  Lengths are post-append (they include the token appended this
 * step).  Every entry a sequence can reach (the first ceil(len / bs) of its
 * row) is checked on the host to be a whole block of `layout` inside the pool,
 * and len <= max_blocks * bs; otherwise KV_ERR_INVALID_ARG and nothing is
 * copied.  Entries past a sequence's last block are not read by any kernel.
 * The copy is a cudaMemcpyAsync from the caller's host buffers: they must stay
 * unchanged until the stream passes this point (pageable memory makes the call
 * synchronous).
 */
int kv_block_table_upload(kv_pool *pool, int layout, const int32_t *host_table, int S,
                          int max_blocks, const int32_t *host_ctx_lens, int32_t *dev_table,
                          int32_t *dev_ctx_lens, void *stream);

/* ------------------------------------------------------ sequence tables --- */

/*
 * A host sequence table of one layout: for each of max_seqs slots, its block
 * list (the row of the block table) and its post-append length.  It carries
 * the runtime's side of the paper's per-stage KV provisioning: a stage
 * reserves ceil((P + L^)/bs) blocks for its predicted total length (Eq. 2),
 * a prediction that falls short grows the reservation one block at a time
 * (a "reservation miss"), a shared prompt prefix is held by reference, and
 * blocks go back to the pool when a stage or sequence ends (§III-C).  Every
 * change is recorded so that kv_seqtab_sync sends only changed table entries
 * to the device.  Not thread-safe; one table per host thread.  A pool
 * destroyed while tables over it are still open detaches them: their blocks
 * end with the pool, every later call on them that would touch a slot
 * returns KV_ERR_INVALID_ARG, and kv_seqtab_destroy only frees the table.
 */
typedef struct kv_seqtab kv_seqtab;

typedef struct kv_seqtab_counters {
    int64_t blocks_held;        /* block references held by all rows */
    int64_t reserve_calls;
    int64_t reservation_misses; /* one-block growths in kv_seq_advance */
    int64_t releases;
    int64_t entries_uploaded;   /* table entries sent by kv_seqtab_sync */
    int64_t sync_launches;
} kv_seqtab_counters;

/* Create an empty table (all lengths 0, all entries -1).  KV_ERR_INVALID_ARG. */
int kv_seqtab_create(kv_pool *pool, int layout, int max_seqs, int max_blocks, kv_seqtab **out);

/* Release every block reference the table holds, then the table. */
int kv_seqtab_destroy(kv_seqtab *t);

/*
 * Make slot s hold at least ceil(tokens / bs) blocks (Eq. 2's reservation
 * for a stage of P + L^ tokens), allocating the missing ones from the pool.
 * All-or-nothing: KV_ERR_OUT_OF_BLOCKS leaves the slot unchanged; more than
 * max_blocks is KV_ERR_INVALID_ARG.
 */
int kv_seq_reserve(kv_seqtab *t, int s, int64_t tokens);

/*
 * Give the empty slot dst the first nblocks blocks of slot src by reference
 * (refcount + 1 each), e.g. a system prompt shared by every agent of a
 * workflow.  The shared blocks must be full (dst's own tokens start at
 * nblocks * bs).  KV_ERR_INVALID_ARG if dst is not empty or src holds fewer.
 */
int kv_seq_share_prefix(kv_seqtab *t, int dst, int src, int nblocks);

/* Set slot s's length (0 .. held blocks * bs).  KV_ERR_INVALID_ARG. */
int kv_seq_set_len(kv_seqtab *t, int s, int32_t len);

/*
 * One decode step for n slots (seqs == NULL: every slot with length > 0):
 * length += 1; a slot whose held blocks are full first grows by one block
 * (a reservation miss).  All-or-nothing over the call: if the pool cannot
 * supply every needed block, KV_ERR_OUT_OF_BLOCKS and nothing changes.
 * *n_grown (may be NULL) receives the number of slots that grew.
 */
int kv_seq_advance(kv_seqtab *t, int n, const int32_t *seqs, int32_t *n_grown);

/* Drop every block reference of slot s and set its length to 0. */
int kv_seq_release(kv_seqtab *t, int s);

/* Drop slot s's reserved blocks beyond ceil(length / bs) (end of a stage). */
int kv_seq_trim(kv_seqtab *t, int s);

/*
 * A step's finished sequences replaced by new admissions, in one call: for
 * i = 0 .. n-1 in order, slot slots[i] drops every block reference it holds
 * (kv_seq_release), then reserves ceil(reserve_tokens[i] / bs) blocks for
 * the new sequence's whole run (Eq. 2) and takes length lens[i]
 * (kv_seq_reserve, kv_seq_set_len).  The release of one slot precedes the
 * next slot's reservation, so freed blocks serve later admissions.
 *   slots          host int32[n], distinct, each in [0, max_seqs)
 *   reserve_tokens host int64[n], 0 .. max_blocks * bs
 *   lens           host int32[n], 0 .. reserve_tokens[i]
 *   status         host int32[n] out: KV_OK, or KV_ERR_OUT_OF_BLOCKS where the
 *                  pool could not serve that reservation (the slot is then
 *                  left empty, length 0, and the admission is the caller's to
 *                  retry); the call itself still returns KV_OK
 * Every argument is checked before any slot changes: KV_ERR_INVALID_ARG and
 * nothing changed.  n = 0 is a no-op.  A failure of the pool itself while
 * slots are replaced (a table naming blocks the pool does not hold live)
 * returns that error at the slot where it occurred; the slots before it
 * stay replaced.
 */
int kv_seq_replace(kv_seqtab *t, int n, const int32_t *slots, const int64_t *reserve_tokens,
                   const int32_t *lens, int32_t *status);

/*
 * Bring a device copy of the table up to date on `stream`: every slot's
 * length goes to dev_ctx_lens[0 .. max_seqs), and every table entry changed
 * since the previous sync (of this table, to any device copy) goes to
 * dev_table (int32 [max_seqs][max_blocks]).  The values travel as kernel
 * parameters, so the host table may change right after the call returns.
 * The first sync after create sends the whole table.  The sync kernel is a
 * programmatic dependent of the previous work in the stream: its launch
 * overlaps that work, and it waits for it to complete before writing.
 */
int kv_seqtab_sync(kv_seqtab *t, int32_t *dev_table, int32_t *dev_ctx_lens, void *stream);

/*
 * Read-only host views: table int32 [max_seqs][max_blocks] (-1 = no block)
 * and lengths int32 [max_seqs]; valid until the next call that changes t.
 */
int kv_seqtab_host(const kv_seqtab *t, const int32_t **table, const int32_t **ctx_lens);

int kv_seqtab_get_counters(const kv_seqtab *t, kv_seqtab_counters *out);

/* ---------------------------------------------------- memory accounting --- */

/*
 * Explicit memory accounting of a node runtime that colocates several models
 * on one GPU (§III-C).  With M_total the GPU memory available to the runtime,
 * M_kv the KV in use and, for every warm model k (Running or Sleeping), its
 * persistent footprint M_ctx^k:
 *     M_res = sum_k M_ctx^k + M_other,   safe iff M_kv + M_res <= M_total,
 * and the KV admission headroom reported to the scheduler is
 *     R_kv^head = M_total - M_res - M_kv.
 * A model's persistent footprint is its kept runtime context (CUDA graphs,
 * compiled kernels, buffers), plus its weights while those are on the GPU.
 * Byte counts are the caller's; these calls touch no device memory.
 */
typedef enum kv_engine_state {
    KV_ENGINE_IDLE = 0,          /* Running, no stage executing: weights + context on the GPU */
    KV_ENGINE_SLEEPING = 1,      /* weights on the host, GPU context kept */
    KV_ENGINE_SLEEP_PENDING = 2, /* a sleep transition has begun: weights + context still on the GPU */
    KV_ENGINE_ACTIVE = 3,        /* Running with executing stages that hold KV */
    KV_ENGINE_COLD = 4           /* CPU-, disk-resident or remote: nothing on the GPU, not warm */
} kv_engine_state;

typedef struct kv_engine {
    int32_t state;             /* kv_engine_state */
    int32_t reserved;          /* 0 */
    uint64_t ctx_bytes;        /* kept runtime context (M_ctx without weights) */
    uint64_t weight_bytes;     /* weights; on the GPU in IDLE, SLEEP_PENDING and ACTIVE */
    uint64_t kv_bytes;         /* KV mapped for the engine's executing stages (ACTIVE only) */
    uint64_t virtual_kv_bytes; /* the engine's virtual KV address space (may exceed physical) */
    double weight_reload_s;    /* time to bring the weights back (profiled bandwidth) */
    double ctx_rebuild_s;      /* time to rebuild the runtime context */
    double kv_swap_in_s;       /* time to swap the engine's KV back in */
    double kv_regen_s;         /* time to regenerate the engine's KV (profiled compute) */
} kv_engine;

typedef struct kv_account {
    uint64_t m_res;            /* sum of warm footprints + M_other */
    uint64_t m_kv;             /* kv_bytes of ACTIVE engines + extra_kv_bytes */
    uint64_t m_kv_virtual;     /* virtual_kv_bytes of warm engines */
    int64_t headroom;          /* R_kv^head = M_total - M_res - M_kv (negative when unsafe) */
    int32_t safe;              /* M_kv + M_res <= M_total */
    int32_t reserved;
    double overcommit;         /* m_kv_virtual / M_total (0 when M_total is 0) */
} kv_account;

/*
 * Account n engines.  extra_kv_bytes adds KV in use that no listed engine
 * owns.  KV_ERR_INVALID_ARG for a null pointer, n < 0 or a bad state.
 */
int kv_memory_account(const kv_engine *engines, int n, uint64_t m_total, uint64_t m_other,
                      uint64_t extra_kv_bytes, kv_account *out);

typedef enum kv_degrade_action {
    KV_ACT_SLEEP = 1,      /* level 1: an idle Running model goes to sleep; frees its weights */
    KV_ACT_EVICT = 2,      /* level 2: a Sleeping model is evicted; frees its context */
    KV_ACT_STOP = 3,       /* level 3: a pending sleep transition is stopped by shutting the
                              engine down; frees weights + context */
    KV_ACT_PREEMPT = 4,    /* level 4: an Active model's KV is swapped out to the host */
    KV_ACT_ABORT = 5       /* level 5: an Active model's executions are aborted; frees their KV */
} kv_degrade_action;

typedef struct kv_plan_step {
    int32_t engine;        /* index into the engines array */
    int32_t action;        /* kv_degrade_action */
    uint64_t freed_bytes;  /* estimated memory the action frees */
    double cost_s;         /* c(e, a): restoration latency of the action */
} kv_plan_step;

/*
 * Minimum-impact memory coordination (Alg. 2) and its disruption cost
 * (Eq. 3).  Warm engines are visited level by level (IDLE, SLEEPING,
 * SLEEP_PENDING, ACTIVE; within a level in array order, so pass them
 * least-recently-used first) and each receives the least disruptive action
 * its state allows, until the freed memory reaches `required` bytes:
 *   IDLE -> SLEEP (frees weights, c = weight_reload_s);
 *   SLEEPING -> EVICT (frees context, c = ctx_rebuild_s);
 *   SLEEP_PENDING -> STOP (frees weights + context, c = weight_reload_s + ctx_rebuild_s);
 *   ACTIVE -> PREEMPT while its KV fits the host swap space the plan has
 *     left (c = kv_swap_in_s), else ABORT (c = kv_regen_s); both free the
 *     KV and raise the interrupt flag.
 * Engines whose action would free nothing, and COLD engines, are passed over.
 *   C_deg = sum over the plan of c(e, a) + [interrupt] * c_int.
 * Up to max_steps steps are written (n_steps counts all of them).  Returns
 * KV_OK when the plan frees at least `required`, KV_ERR_OUT_OF_BLOCKS
 * (infeasible: every engine was used and still less was freed; the steps
 * are still written), KV_ERR_INVALID_ARG for bad arguments.  required = 0
 * gives an empty plan with C_deg = 0.
 */
int kv_degradation_plan(const kv_engine *engines, int n, uint64_t required, uint64_t host_swap_bytes,
                        double c_int, kv_plan_step *steps, int max_steps, int *n_steps, int *interrupt,
                        double *c_deg, uint64_t *freed);

/*
 * Admission check of a stage that needs `demand` more bytes of KV (§III-C).
 * If demand <= R_kv^head the stage fits: KV_OK with *n_steps = 0 and
 * C_deg = 0.  Otherwise a degradation plan for R = demand - R_kv^head is
 * derived as kv_degradation_plan does: KV_OK with *n_steps > 0 when the plan
 * makes room (the caller executes it before admitting), KV_ERR_OUT_OF_BLOCKS
 * when it cannot (the stage is rejected; the plan and C_deg still describe
 * everything the node could free).  *headroom receives R_kv^head before any
 * degradation.
 */
int kv_admission_check(const kv_engine *engines, int n, uint64_t m_total, uint64_t m_other,
                       uint64_t extra_kv_bytes, uint64_t demand, uint64_t host_swap_bytes, double c_int,
                       kv_plan_step *steps, int max_steps, int *n_steps, int *interrupt, double *c_deg,
                       int64_t *headroom);

/* -------------------------------------------------------------- kernels --- */

/*
 * Append one token per sequence (the decode step writes the new token's K/V
 * before attending, §II): for s < S with n = dev_ctx_lens[s] > 0 and every KV
 * head g, copy k_new[s][g][:] and v_new[s][g][:] (bf16 [S][Hkv][d] device
 * arrays) bit-exactly into slot (table[s][(n-1)/bs], (n-1) % bs).  Sequences
 * with n <= 0 are skipped.  Device bounds failures skip the row and set the
 * error word.
 */
int kv_append(kv_pool *pool, int layout, const uint16_t *k_new, const uint16_t *v_new,
              const int32_t *dev_table, const int32_t *dev_ctx_lens, int max_blocks, int S,
              void *stream);

/*
 * Bytes of device workspace paged_decode_attn needs for these sizes and this
 * num_splits: one (first part, part count) pair of int32 per (sequence, KV
 * head) run, followed by fp32 split partials, one record of G*d + 2*G floats
 * per (run, part) pair a split run can produce.  Every call writes all it reads, so the
 * workspace needs no initialisation and may be reused freely by calls that
 * are ordered on one stream.
 */
int kv_workspace_bytes(const kv_pool *pool, int layout, int S, int Hq, int max_blocks,
                       int num_splits, size_t *out_bytes);

/* Zero a workspace on `stream` (cudaMemsetAsync); not required before use. */
int kv_workspace_clear(void *workspace, size_t ws_bytes, void *stream);

/*
 * Batched paged decode attention.  For every sequence s < S (post-append
 * length n = dev_ctx_lens[s]), every query head h < Hq and its KV head
 * g = floor(h / G), G = Hq / Hkv (contiguous head groups):
 *     out[s][h] = sum_{j<n} softmax_j(scale * q[s][h] . K_j) V_j
 * with K_j, V_j the rows of head g at position j, found through dev_table.
 * q, out: bf16 [S][Hq][d] arrays, 16-byte aligned, in device memory or in
 * pinned (page-locked, mapped) host memory: the kernels read q with
 * 16-byte copies into shared memory (cp.async) and write out with ordinary
 * stores, which on GB300 cross the coherent NVLink-C2C link to host
 * memory, so a caller holding a step's inputs and
 * results on the host needs no separate copies (the same holds for k_new
 * and v_new of the calls below).  The pool, table, lengths and workspace
 * are device memory.  A sequence with n == 0 gets zeros.
 * Arithmetic: fp32 products and accumulation, online softmax in base 2,
 * bf16 output rounded to nearest-even.
 * Work split: the batch's KV is cut into 16-token tiles of one (sequence,
 * KV head); the tiles are split into equal contiguous parts, one per warp of
 * the resident CTAs (num_splits == 0), or into num_splits * 8 parts when
 * num_splits > 0 CTAs are requested.  A (sequence, head) whose tiles fall in
 * more than one part leaves fp32 partials (max, sum, unnormalised output)
 * that a second kernel merges in part order, so results do not depend on
 * where blocks sit in the pool.  Launches two kernels on `stream`.
 * Errors: KV_ERR_INVALID_ARG, KV_ERR_UNSUPPORTED (d not 64/128, G not in
 * {1,2,4,5,8}, block size not a multiple of 16), KV_ERR_WORKSPACE.
 */
int paged_decode_attn(kv_pool *pool, int layout, const uint16_t *q, uint16_t *out,
                      const int32_t *dev_table, const int32_t *dev_ctx_lens, int max_blocks,
                      int S, int Hq, float scale, int num_splits, void *workspace,
                      size_t ws_bytes, void *stream);

/*
 * kv_append and paged_decode_attn in one pass (one launch fewer per step).
 * The results are those of kv_append(k_new, v_new) followed by
 * paged_decode_attn: the pool afterwards holds each sequence's new row at
 * position n-1, and the attention uses it.  The warp that reads the tile
 * holding position n-1 substitutes the new row in shared memory and then
 * stores it to the pool, so no other reader sees the slot half-written.
 * Sequences with n <= 0 or n beyond the table are not appended to.
 * k_new, v_new: bf16 [S][Hkv][d] device arrays, 16-byte aligned.
 */
int paged_decode_attn_append(kv_pool *pool, int layout, const uint16_t *q, const uint16_t *k_new,
                             const uint16_t *v_new, uint16_t *out, const int32_t *dev_table,
                             const int32_t *dev_ctx_lens, int max_blocks, int S, int Hq, float scale,
                             int num_splits, void *workspace, size_t ws_bytes, void *stream);

/*
 * kv_seqtab_sync(t, dev_table, dev_ctx_lens, stream) followed by
 * paged_decode_attn_append (k_new, v_new given) or paged_decode_attn (both
 * NULL) over the table's first S rows, with layout and max_blocks taken from
 * the table, in one launch when it fits: when the table's lengths and its
 * changed entries since the last sync make at most 128 words, they travel
 * as parameters of the decode kernel, which reads them from there and
 * writes them to dev_ctx_lens / dev_table for later kernels (the separate
 * sync kernel, its hand-off and a dependent read of the lengths drop out of
 * the step).  Otherwise (the first sync, larger batches or many changes)
 * the call runs kv_seqtab_sync and then the plain call.  Results, device
 * table and lengths afterwards are those of the two calls; errors are theirs
 * (KV_ERR_INVALID_ARG also when t is not over `pool` or S > max_seqs).
 */
int paged_decode_attn_seqtab(kv_pool *pool, kv_seqtab *t, const uint16_t *q, const uint16_t *k_new,
                             const uint16_t *v_new, uint16_t *out, int32_t *dev_table, int32_t *dev_ctx_lens,
                             int S, int Hq, float scale, int num_splits, void *workspace, size_t ws_bytes,
                             void *stream);

/*
 * Several decode batches in one call: co-located models, each with its own
 * layout, queries, tables and workspace, attending over the one pool.  The
 * result is that of calling paged_decode_attn (k_new / v_new NULL) or
 * paged_decode_attn_append for batches[0], batches[1], ... in order, with
 * num_splits = 0.  The decode kernels run as a chain: each later batch's
 * kernel starts on the SMs the one before frees as its last warps finish,
 * and the split-K merges of all batches follow.  Batches must not share a
 * workspace or an output, and no batch may read a block that another one
 * appends to (blocks of different layouts never overlap).  All arguments
 * are checked before anything is launched; errors are those of
 * paged_decode_attn.  Batches with S = 0 are skipped.
 */
typedef struct kv_attn_batch {
    int layout;
    const uint16_t *q;      /* [S][Hq][d] */
    const uint16_t *k_new;  /* [S][Hkv][d] or NULL (no append) */
    const uint16_t *v_new;  /* [S][Hkv][d] or NULL */
    uint16_t *out;          /* [S][Hq][d] */
    const int32_t *dev_table;
    const int32_t *dev_ctx_lens;
    int max_blocks;
    int S;
    int Hq;
    float scale;
    void *workspace;        /* kv_workspace_bytes(pool, layout, S, Hq, max_blocks, 0) */
    size_t ws_bytes;
} kv_attn_batch;

int paged_decode_attn_multi(kv_pool *pool, int n, const kv_attn_batch *batches, void *stream);

/*
 * Shared-prefix ("cascade") decode attention.  Sequences that hold the same
 * physical blocks at the start of their block tables -- a system prompt
 * shared by reference by every stage of an agent workflow (§III-B, §III-C)
 * -- have identical K/V for those tokens.  For every group of such
 * sequences, the prefix's attention is computed once per KV head for all
 * members together as a dense tensor-core contraction, each member's own
 * suffix is streamed as in paged_decode_attn (with the fused append when
 * k_new / v_new are given, as paged_decode_attn_append), and the two are
 * merged exactly (the softmax factorises over a partition of the keys).
 * The result equals paged_decode_attn's on the same inputs, up to rounding.
 *
 * groups[i] = {count, tokens}: group i's members are the next `count`
 * entries of members[] (host arrays, groups in order); `tokens` is the
 * shared prefix length, a multiple of 64 and of the block size, at most
 * max_blocks * bs.  The prefix blocks are read from the first member's
 * table row; the caller guarantees every member's first tokens/bs entries
 * are the same blocks and, when appending, that every member's length
 * (post-append) exceeds tokens (so the new token never lands in a shared
 * block).  A member whose length equals tokens (no append) attends over the
 * prefix alone.  A sequence is in at most one group; sequences in no group
 * are computed as by paged_decode_attn.  n_groups = 0 is paged_decode_attn
 * (or _append).  The plan travels as a kernel's parameters and then in
 * the workspace:
 *     3 * n_groups + 2 + (members) + S <= 4080 words.
 * Workspace: kv_cascade_workspace_bytes() (256-byte aligned); nothing in it
 * needs initialising.  Consecutive calls on one workspace alternate between
 * its two skip arrays (step overlap, kv_set_attn_step_overlap).
 * Errors: KV_ERR_INVALID_ARG (bad plan, duplicate member, words over the
 * limit), KV_ERR_WORKSPACE, KV_ERR_UNSUPPORTED, KV_ERR_CUDA; on the device a
 * member shorter than its prefix sets KV_ERR_DEVICE_BOUNDS in the error word.
 */
typedef struct kv_prefix_group {
    int32_t count;   /* members in the group */
    int32_t tokens;  /* shared prefix tokens */
} kv_prefix_group;

int kv_cascade_workspace_bytes(const kv_pool *pool, int layout, int S, int Hq, int max_blocks, size_t *out_bytes);

int paged_decode_attn_cascade(kv_pool *pool, int layout, const uint16_t *q, const uint16_t *k_new,
                              const uint16_t *v_new, uint16_t *out, const int32_t *dev_table,
                              const int32_t *dev_ctx_lens, int max_blocks, int S, int Hq, float scale,
                              const kv_prefix_group *groups, int n_groups, const int32_t *members, void *workspace,
                              size_t ws_bytes, void *stream);

/*
 * kv_seqtab_sync(t, dev_table, dev_ctx_lens, stream) followed by
 * paged_decode_attn_cascade over the table's first S rows (layout and
 * max_blocks taken from the table), with the sync carried by the cascade
 * call's first launch: when the plan's words, the table's S lengths and
 * two words per entry changed since the last sync make at most 4080 words,
 * the kernel that writes the plan to the workspace also writes the lengths
 * and the changed entries to dev_ctx_lens / dev_table (the separate sync
 * kernel and its hand-off drop out of the step).  Otherwise (the first
 * sync, or more changes than fit) the call runs kv_seqtab_sync first.
 * n_groups = 0 is paged_decode_attn_seqtab with num_splits = 0; S = 0 is
 * kv_seqtab_sync alone.  Results, device table and lengths afterwards are
 * those of the two calls; errors are theirs (KV_ERR_INVALID_ARG also when t
 * is not over `pool` or S > max_seqs).
 */
int paged_decode_attn_cascade_seqtab(kv_pool *pool, kv_seqtab *t, const uint16_t *q, const uint16_t *k_new,
                                     const uint16_t *v_new, uint16_t *out, int32_t *dev_table,
                                     int32_t *dev_ctx_lens, int S, int Hq, float scale,
                                     const kv_prefix_group *groups, int n_groups, const int32_t *members,
                                     void *workspace, size_t ws_bytes, void *stream);

/*
 * paged_decode_attn for callers that cannot allocate device memory.  The
 * paper has no counterpart; this is a service of this library.  Callers that
 * cannot hand over a workspace include a server whose KV pool already holds
 * all free HBM, a host framework whose allocator this layer may not call,
 * and a decode loop in which a cudaMalloc (which may synchronise the whole
 * device) is not acceptable.
 * Arguments and results are those of paged_decode_attn without the
 * workspace.  The split-K scratch is instead a fixed 32 MiB device array
 * inside the library, held on a device until the process exits once it has
 * been taken there.  The call allocates nothing.
 *   - Creating a pool (kv_pool_create, kv_pool_create_vmm) looks up the
 *     array's device address (cudaGetSymbolAddress) with the pool's device
 *     current.  CUDA loads modules lazily by default, so that lookup is when
 *     the 32 MiB are taken from the device: before the caller fills the
 *     device with KV blocks.  If it failed there, the first call on the
 *     device repeats it, and then needs the 32 MiB free.  Create the pool
 *     before any stream capture.
 *   - The pool's device must be the current device (else
 *     KV_ERR_INVALID_ARG, nothing launched): each device has its own array.
 *   - If kv_workspace_bytes for the same arguments exceeds 32 MiB the call
 *     returns KV_ERR_WORKSPACE and launches nothing; use paged_decode_attn
 *     with a workspace for such batches.
 *   - Every call uses the same array, which keeps the last call's contents.
 *     Nothing in it has to start at zero (each call writes what it reads),
 *     but calls that can overlap on the GPU (streams with no ordering
 *     between them) race on it; calls on one stream are ordered.
 */
int paged_decode_attn_noalloc(kv_pool *pool, int layout, const uint16_t *q, uint16_t *out,
                              const int32_t *dev_table, const int32_t *dev_ctx_lens, int max_blocks,
                              int S, int Hq, float scale, int num_splits, void *stream);

/*
 * Select the attention compute variant for later calls on this pool:
 * 0 = automatic (the fastest measured for the shape), 1 = CUDA-core FMA,
 * 2 = warp-level tensor-core MMA (mma.sync bf16, fp32 accumulate).
 */
int kv_set_attn_variant(kv_pool *pool, int variant);

/*
 * Step overlap for later attention calls on this pool (0 = off, the
 * default; 1 = on).  On, a paged_decode_attn, paged_decode_attn_append or
 * paged_decode_attn_seqtab call (and the allocation-free call) whose stream
 * last received, from this library, the split-K combine of an earlier
 * attention call starts its decode kernel while that combine is still
 * finishing: the decode kernel reads the lengths, the table and the pool
 * and starts streaming at once, and waits for the combine before it writes
 * the output or the workspace.  That is safe because the combine releases
 * the next kernel only after everything before it in the stream has
 * completed.  A shared-prefix call (paged_decode_attn_cascade,
 * paged_decode_attn_cascade_seqtab) overlaps the combine of the previous
 * shared-prefix call when that call used the same workspace with the same
 * layout: its plan kernel writes the plan, the skips (into the workspace's
 * other skip array) and the table sync at once and raises a flag in the
 * workspace; the decode kernel over the suffixes, released by the prefix
 * kernel before that kernel's own wait, reads after that flag and writes
 * its output and partials after a second flag, which the plan kernel
 * raises once the combine has completed.  Any other launch or copy of this
 * library on the stream in between (a table sync, an append, an upload)
 * turns it off for the next call, and so does a stream the library has not
 * seen.  Results are the same bits either way; kv_pool_stats counts the
 * calls that overlapped.  The caller's side of the contract: work of
 * others between two attention calls on one stream must not be launched as
 * a programmatic dependent that releases its own dependents before it has
 * finished writing (ordinary kernels and copies are fine); one host thread
 * submits to the stream at a time; and the earlier call's workspace and
 * output are not handed to the later call as its table, lengths or inputs
 * (a stream-ordered allocator that reuses freed memory on the same stream
 * at once can do that when they are freed between the calls).
 */
int kv_set_attn_step_overlap(kv_pool *pool, int on);

/* Library version string (static storage). */
const char *kv_version(void);

#ifdef __cplusplus
}
#endif

#endif /* KVPOOL_H */
