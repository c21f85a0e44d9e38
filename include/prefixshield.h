/*
 * prefixshield.h -- C ABI of the GB300 (sm_103a) batched prefix-cache step of
 * PrefixShield (Wang and Buyya, "Preserving Admission Responsibility in
 * Multi-Tenant Large Language Model Prefix Caches", arXiv 2608.01657).
 *
 * One handle owns one shared, multi-tenant pool of KV blocks (one replacement
 * domain, Sec. II-C).  Each ps_step() processes one batch of requests in five
 * stages, all on the GPU, asynchronously on the caller's stream:
 *   1. chained hashing of every full block of every prompt (Sec. III-B);
 *   2. longest-cached-prefix lookup, namespace-scoped by accounting group
 *      (n_cached of Alg. 1);
 *   3. metering of newly materialized full blocks into per-(group, contract)
 *      token buckets with lazy refill (Eq. 1-3, OnCacheFullBlocks of Alg. 1);
 *   4. debt-gated reuse promotion (Eq. 4, OnTouch of Alg. 1);
 *   5. reclamation: true-free blocks first, then victims chosen by projected
 *      normalized debt and retention segment (Eq. 5-9, Alg. 2), or by the LRU
 *      or S3-FIFO baselines (Sec. V-A).
 *
 * Conventions shared by every entry point:
 *  - Pointers named d_* are device pointers on the device that was current at
 *    ps_create(); h_* are host pointers.  The caller owns every buffer,
 *    including the device workspace; the library never allocates device
 *    memory.  ps_create() allocates only the small host-side handle.
 *  - Streams are passed as void* holding a cudaStream_t (NULL = legacy stream).
 *  - Every call returns an int32 status (PS_OK = 0, errors < 0).  Errors the
 *    host can see (bad sizes, null pointers, capacities) are returned before
 *    any work is enqueued.  Errors only the device can see (bad offsets or
 *    group ids, a clock that goes backwards) make that step a no-op that
 *    leaves all state unchanged and report the code in out->counts[3].
 *    Running out of prefix-history capacity (a step that would hold more
 *    than history_capacity distinct (group, prefix id) entries) also leaves
 *    all state unchanged, and is sticky: every later step is a no-op
 *    reporting PS_ERR_CAPACITY until ps_clear_status() or ps_reset().
 *  - A handle is not thread-safe; steps on one handle must be issued in
 *    order on one stream (or with equivalent ordering).
 */
#ifndef PREFIXSHIELD_H
#define PREFIXSHIELD_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

#define PS_MAX_CONTRACTS 8
#define PS_MAX_GROUPS 1024
#define PS_NUM_STATS 15
/* Limits of one step (a step with more is rejected as PS_ERR_INVALID_ARG);
 * after 2^31 - 1 steps a handle reports PS_ERR_CAPACITY until ps_reset(). */
#define PS_MAX_REQUESTS_PER_STEP ((1 << 18) - 1)
#define PS_MAX_BLOCKS_PER_REQUEST ((1 << 18) - 1)

typedef enum {
  PS_LRU = 0,          /* global recency (vLLM free queue), Sec. V-A */
  PS_S3FIFO = 1,       /* S3-FIFO baseline, Sec. V-A */
  PS_PREFIXSHIELD = 2, /* Alg. 1 + Alg. 2 */
  PS_STATICQUOTA = 3   /* equal per-group partitions of floor(N / G) blocks, no
                          borrowing; recency inside a partition (Sec. V-A) */
} ps_policy_t;

enum {
  PS_OK = 0,
  PS_ERR_INVALID_ARG = -1,
  PS_ERR_CAPACITY = -2,
  PS_ERR_CLOCK = -3,
  PS_ERR_CUDA = -4,
  PS_ERR_TIMEOUT = -5,
  PS_ERR_DEVICE_STATUS = -6
};

#define PS_FLAG_NO_SEGMENTATION 1u /* ablation: victims inside a group by recency only */
#define PS_FLAG_NO_DEBT_GATE 2u    /* ablation: promote regardless of debt (Eq. 4 off) */
/* Victim selection from indexed per-(group, class) queues (the indexed
 * per-group, per-segment queues Sec. VIII proposes) instead of a scan of
 * every candidate.  Same victims, same results; lru, prefixshield and
 * staticquota (ignored for s3fifo, which keeps its own queues).  The
 * workspace grows by two buffers of 16 x (N + max_tokens / block_size)
 * entries of 12 bytes each, plus per-step scratch. */
#define PS_FLAG_INDEXED_QUEUES 4u
/* With PS_FLAG_INDEXED_QUEUES: the first scan round of a take covers a single
 * 1024-entry chunk, so a take that needs more finishes in the second round.
 * Same results, slower; it exercises the second round on small pools. */
#define PS_FLAG_QUEUE_SHORT_WINDOWS 8u
/* With s3fifo: the ghost FIFO's live entries are compacted into its second
 * ring on every step that has any (normally only when the ring lacks room for
 * the step's pushes).  Same results, slower; it exercises the compaction on
 * small pools. */
#define PS_FLAG_S3_COMPACT_GHOST 16u
/* With s3fifo: every step's evictions run the published one-at-a-time loop on
 * one device thread instead of the closed form computed in parallel (which
 * falls back to that loop only where it does not apply).  Same results,
 * slower; it checks the sequential kernel over whole traces. */
#define PS_FLAG_S3_SEQUENTIAL 32u

/* Per-group statistics, int64 each, row-major [num_groups][PS_NUM_STATS]. */
enum {
  PS_STAT_REQUESTS = 0,       /* requests of the group */
  PS_STAT_PROMPT_TOKENS,      /* prompt tokens, full blocks or not */
  PS_STAT_FULL_BLOCKS,        /* full blocks n_full */
  PS_STAT_HIT_BLOCKS,         /* cached prefix + in-step hits */
  PS_STAT_INSTEP_HIT_BLOCKS,  /* hits on blocks materialized earlier in the same step */
  PS_STAT_HIT_TOKENS,         /* block_size * hit blocks (cached_tokens, Sec. V-A) */
  PS_STAT_ADMITTED_BLOCKS,    /* newly materialized = charged blocks n_r (I1) */
  PS_STAT_UNGRANTED_BLOCKS,   /* claims the pool could not hold this step */
  PS_STAT_EVICTED_BLOCKS,     /* reclaimed blocks owned by the group */
  PS_STAT_INVALIDATED_BLOCKS, /* orphaned blocks dropped (parent was reclaimed) */
  PS_STAT_PROMOTIONS,         /* blocks promoted to Reuse (Eq. 4) */
  PS_STAT_GATED_REUSES,       /* proven reuses refused by the debt gate */
  PS_STAT_RESIDENT_BLOCKS,    /* current occupancy */
  PS_STAT_DEBT_RAW,           /* D_g after the last step, fixed point (Eq. 3) */
  PS_STAT_DEBT_NORM           /* normalized debt after the last step (Eq. 5) */
};

/* Policy parameters.  Rates and balances are in blocks scaled by 2^fp_shift. */
typedef struct {
  int32_t num_contracts;                       /* C, 1..PS_MAX_CONTRACTS */
  int32_t fp_shift;                            /* fixed-point scale, 0..30 (default 20) */
  int64_t epsilon_fp;                          /* debt tolerance epsilon >= 0 (Sec. III-B) */
  int64_t rho_fp[PS_MAX_CONTRACTS];            /* refill per accounting tick rho_c > 0 (Eq. 1) */
  int64_t beta_fp[PS_MAX_CONTRACTS];           /* burst capacity beta_c >= 0 (Eq. 1) */
  int32_t contract_of_group[PS_MAX_GROUPS];    /* contract used when a step passes no contract ids */
  uint64_t hash_seed;                          /* seed of the block-key function */
  int32_t s3_small_pct;                        /* S3-FIFO small queue, percent of the pool (10) */
  /* S3-FIFO counter cap (3: a two-bit counter).  A step's evictions run in
   * parallel in closed form for caps up to 15; caps of 16 or more, and steps
   * whose main queue would run empty (common when the small queue is near
   * 100% of the pool), take the one-at-a-time loop on one device thread:
   * the same results, much slower on large pools. */
  int32_t s3_freq_cap;
  int32_t s3_move_min_freq;                    /* small->main when freq >= this (2) */
  int32_t pad0;
  int64_t history_capacity;                    /* max distinct (group, prefix id) entries */
  uint32_t flags;                              /* PS_FLAG_* */
  uint32_t pad1;
} ps_params_t;

/* Outputs of one step, all device pointers, caller-owned.  R = num_requests,
 * B = max_tokens / block_size (the handle's per-step block capacity).  A step
 * can write up to B ids into each id list (the lists' lengths are known only
 * on the device), so each must hold B: ids_capacity (elements in each of the
 * three id arrays) below B, or req_capacity (elements in hit_blocks and
 * admitted_blocks; admitted_offsets holds one more) below R, is refused with
 * PS_ERR_INVALID_ARG before anything is enqueued.  The arrays' real sizes
 * are the caller's to state truthfully: the library cannot check pointers. */
typedef struct {
  int32_t* hit_blocks;        /* [R]   cached prefix + in-step hits of each request */
  int32_t* admitted_blocks;   /* [R]   newly materialized (charged) blocks n_r */
  int32_t* admitted_offsets;  /* [R+1] CSR offsets into admitted_ids */
  int32_t* admitted_ids;      /* [B]   block ids, request-major then position order */
  int32_t* evicted_ids;       /* [B]   reclaimed block ids, ascending */
  int32_t* invalidated_ids;   /* [B]   orphaned block ids dropped, ascending */
  int32_t* counts;            /* [4]   n_admitted, n_evicted, n_invalidated, step status */
  int64_t* debt_raw;          /* [G]   D_g after the step (Eq. 3) */
  int64_t* debt_norm;         /* [G]   normalized debt after the step (Eq. 5) */
  int64_t ids_capacity;       /* elements in each of admitted_ids, evicted_ids, invalidated_ids (>= B) */
  int32_t req_capacity;       /* elements in hit_blocks and admitted_blocks (>= R) */
  int32_t pad;
} ps_step_out_t;

/* Host-side copy of a step's outputs for ps_step_host(); same layout. */
typedef ps_step_out_t ps_host_out_t;

typedef struct ps_handle ps_handle_t;

/* Bytes of device workspace a handle needs (256-byte aligned base required),
 * or 0 if the arguments are invalid.  Arguments as for ps_create(). */
size_t ps_workspace_bytes(int64_t capacity_blocks, int32_t block_size, int32_t num_groups,
                          const ps_params_t* params, int32_t max_requests, int64_t max_tokens);

/* Create a pool of capacity_blocks blocks (all free, every balance full:
 * B = beta at t = 0, Sec. III-B) inside the caller's workspace, and
 * initialize it on 'stream'.  block_size: tokens per KV block, one of 2, 4, 8,
 * 16, 32, 64 (16 in the paper).  max_requests / max_tokens bound every later step.
 * The workspace must stay allocated and untouched until ps_destroy().
 * Returns PS_ERR_INVALID_ARG for bad arguments or a workspace that is too
 * small or misaligned. */
int32_t ps_create(ps_handle_t** out, int64_t capacity_blocks, int32_t block_size, int32_t num_groups,
                  int32_t policy, const ps_params_t* params, void* d_workspace, size_t workspace_bytes,
                  int32_t max_requests, int64_t max_tokens, void* stream);

/* One batched prefix-cache step at accounting time now_ticks (non-decreasing
 * across steps).  Request i has group d_group_ids[i] and the tokens
 * d_tokens[d_token_offsets[i] .. d_token_offsets[i+1]) (int32 ids, offsets
 * start at 0 and do not decrease).  d_contract_ids (nullable) selects each
 * request's service contract, else contract_of_group; d_prefix_ids (nullable,
 * non-zero) gives each request's logical prefix id p, else p is the key of its
 * first full block.  Enqueued on 'stream'; returns without synchronizing. */
int32_t ps_step(ps_handle_t* h, void* stream, int64_t now_ticks, int32_t num_requests,
                const int32_t* d_group_ids, const int64_t* d_token_offsets, const int32_t* d_tokens,
                const int32_t* d_contract_ids, const uint64_t* d_prefix_ids, const ps_step_out_t* out);

/* The same step from host buffers: copies the inputs into the workspace's
 * staging area, runs ps_step(), copies every output back into the caller's
 * host buffers (h_out has the layout of ps_step_out_t with host pointers; the
 * id lists receive only their counts' worth), and synchronizes 'stream'.
 * Pinned host memory makes the copies asynchronous. */
int32_t ps_step_host(ps_handle_t* h, void* stream, int64_t now_ticks, int32_t num_requests,
                     const int32_t* h_group_ids, const int64_t* h_token_offsets, const int32_t* h_tokens,
                     const int32_t* h_contract_ids, const uint64_t* h_prefix_ids, const ps_host_out_t* h_out);

/* Pipelined form of ps_step_host(): enqueue one step from host buffers and
 * return at once, so that the next step's input copy overlaps this step's
 * work.  Two steps may be in flight, on staging slots 0 and 1 (use them in
 * turn; a slot is reused only after ps_step_host_wait() on it).  The inputs
 * are copied on the handle's own copy stream into the slot's staging area
 * (pinned host memory keeps that asynchronous; the buffers must stay
 * unchanged until the wait).  The step itself runs on 'stream', in order with
 * the caller's other work there.  The outputs are written by a kernel
 * directly into h_out, whose non-null arrays must be page-locked host memory
 * (device-accessible; else PS_ERR_INVALID_ARG); the id lists receive only
 * their counts' worth.  Returns PS_OK or a launch error; the step's own
 * status comes from ps_step_host_wait(). */
int32_t ps_step_host_async(ps_handle_t* h, void* stream, int32_t slot, int64_t now_ticks, int32_t num_requests,
                           const int32_t* h_group_ids, const int64_t* h_token_offsets, const int32_t* h_tokens,
                           const int32_t* h_contract_ids, const uint64_t* h_prefix_ids, const ps_host_out_t* h_out);

/* Block until the step enqueued on 'slot' by ps_step_host_async() has
 * written its outputs; returns that step's status (h_out counts[3]). */
int32_t ps_step_host_wait(ps_handle_t* h, int32_t slot);

/* Copy the per-group statistics into h_stats [num_groups][PS_NUM_STATS];
 * synchronizes 'stream'.  Returns the sticky status (PS_OK or PS_ERR_CAPACITY). */
int32_t ps_stats(ps_handle_t* h, void* stream, int64_t* h_stats);

/* Clear a sticky capacity error without resetting the pool (enqueued).  The
 * failed step left no trace, so the next step continues from the state before
 * it; a step that again needs more history entries than the capacity fails
 * again (and is sticky again). */
int32_t ps_clear_status(ps_handle_t* h, void* stream);

/* Return the pool to its state right after ps_create() (enqueued). */
int32_t ps_reset(ps_handle_t* h, void* stream);

/* Free the host-side handle.  The workspace is the caller's to free. */
void ps_destroy(ps_handle_t* h);

const char* ps_status_string(int32_t status);

/* Test hook: copy the full policy state to host arrays (synchronizes).
 * Per block [capacity_blocks]: resident, key, group, contract, prefix id,
 * retention class (0 Probationary, 1 Normal, 2 Reuse), recency stamp, access
 * count, S3-FIFO frequency (capped) / queue (0 small, 1 main) / sequence.
 * Ledger [num_groups * num_contracts] balances; scalars: last refill tick,
 * next step index, S3-FIFO and ghost sequence counters.  Any pointer may be
 * NULL to skip that array.  Fields of non-resident blocks are unspecified. */
typedef struct {
  uint8_t* resident; uint64_t* key; int32_t* group; int32_t* contract; uint64_t* prefix;
  int32_t* klass; uint64_t* stamp; uint32_t* acc; int32_t* freq; int32_t* s3q; uint64_t* s3seq;
  int64_t* balances;
  int64_t t_prev; uint64_t step; uint64_t s3_ctr; uint64_t ghost_ctr;
} ps_state_view_t;
int32_t ps_export_state(ps_handle_t* h, void* stream, ps_state_view_t* h_view);

/* Test hook: live prefix-history entries (group, prefix id, reference count,
 * admitted flag), unordered.  With NULL arrays returns the count only;
 * otherwise fills at most 'cap' entries and returns the count.  Synchronizes. */
int64_t ps_export_history(ps_handle_t* h, void* stream, int32_t* h_group, uint64_t* h_prefix,
                          uint64_t* h_refcount, uint8_t* h_admitted, int64_t cap);

/* Test hook: live S3-FIFO ghost entries (group, key, sequence), unordered;
 * same convention as ps_export_history. */
int64_t ps_export_ghost(ps_handle_t* h, void* stream, int32_t* h_group, uint64_t* h_key, uint64_t* h_seq,
                        int64_t cap);

/* Read-only probe of the cache: for each request, the number of leading full
 * blocks of its prompt resident in the pool now (n_cached of Alg. 1 as
 * ps_step() would find it before any request of the batch materializes a
 * block).  Nothing in the pool changes.  Arguments as for ps_step();
 * d_cached_blocks [R] receives the counts and d_status (device int32) the
 * outcome: PS_OK, or PS_ERR_INVALID_ARG for bad offsets or group ids or more
 * than max_tokens tokens.  Uses the handle's workspace as scratch: do not run
 * it concurrently with a ps_step() of the same handle.  Enqueued on 'stream'. */
int32_t ps_cached_prefix(ps_handle_t* h, void* stream, int32_t num_requests, const int32_t* d_group_ids,
                         const int64_t* d_token_offsets, const int32_t* d_tokens, int32_t* d_cached_blocks,
                         int32_t* d_status);

/* ps_cached_prefix() for callers that cannot allocate device memory.  The
 * paper has no counterpart: this is a deployment convenience.  Some callers
 * may not call cudaMalloc or write into a workspace they do not own -- code
 * inside a CUDA graph capture region, or code under a framework whose
 * allocator owns every device allocation.  This variant computes the same
 * counts as ps_cached_prefix() with its scratch in one fixed array compiled
 * into the library (about 2.4 MB, held on every GPU that loads the library
 * until the process exits).  It allocates nothing; the caller passes inputs
 * and outputs as for ps_cached_prefix().  Only the scratch leaves the
 * workspace: the probe reads the pool's table, which every ps_step() of the
 * handle rewrites, so it must be ordered on the GPU (same stream, or events)
 * against every ps_step() of that handle.  Limits of one call: the handle's
 * max_requests (more returns PS_ERR_INVALID_ARG, as ps_cached_prefix()
 * does), 4096 requests (more returns PS_ERR_CAPACITY at once), and 131072
 * full blocks (more tokens than 131072 * block_size make d_status
 * PS_ERR_INVALID_ARG).  The first call on a device looks up the array's
 * device address for that device; make that first call before any stream
 * capture.  Every call on a device shares the one array: calls that overlap
 * on the GPU (other streams, other handles, other threads) race and must be
 * serialized by the caller. */
int32_t ps_cached_prefix_noalloc(ps_handle_t* h, void* stream, int32_t num_requests, const int32_t* d_group_ids,
                                 const int64_t* d_token_offsets, const int32_t* d_tokens, int32_t* d_cached_blocks,
                                 int32_t* d_status);

/* Profiling hook.  When enabled, ps_step() records a CUDA event on its
 * stream before each of its PS_NUM_STAGES stages and after the last one:
 *   0 validate, 1 hash + lookup, 2 claims + orphans, 3 grant + in-step hits,
 *   4 metering, 5 touch + gate, 6 victim selection, 7 free-take + id lists,
 *   8 eviction (empty: each victim's old content is dropped by the insertion
 *   that reuses its id), 9 eviction + insertion, 10 commit.
 * Creating the events is the only work; no device memory is allocated. */
#define PS_NUM_STAGES 11
int32_t ps_set_stage_timing(ps_handle_t* h, int32_t enable);

/* Per-stage durations in milliseconds of the last timed step (synchronizes on
 * its last event).  Writes min(max_stages, PS_NUM_STAGES) values and, if
 * h_launches is not NULL, the number of kernels that step launched.  Returns
 * the number of stages written, or an error. */
int32_t ps_get_stage_times(ps_handle_t* h, float* h_ms, int32_t max_stages, int32_t* h_launches);

/* 1 if the handle replays its step as one captured CUDA graph (the step's
 * per-call arguments live in a device block that every kernel reads, so one
 * graph serves every step; phases many steps skip are conditional nodes), 0
 * if it launches kernel by kernel (the graph could not be captured or
 * instantiated: results are the same).  Known after the first ps_step().
 * Measurement hook; the paper has no counterpart. */
int32_t ps_uses_graph(const ps_handle_t* h);

/* Launch mode of ps_step(): enable = 1 (the default) replays the step as one
 * captured CUDA graph, enable = 0 launches its kernels one by one on the
 * caller's stream (for profilers that cannot see inside graphs with
 * conditional nodes).  The same kernels do the same work either way.
 * Measurement hook; the paper has no counterpart. */
int32_t ps_set_graph(ps_handle_t* h, int32_t enable);

#ifdef __cplusplus
}
#endif

#endif /* PREFIXSHIELD_H */
