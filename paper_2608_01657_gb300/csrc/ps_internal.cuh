// Internal declarations of the GB300 prefix-cache step library.
//
// Device state lives in one caller-provided workspace, carved into the
// structure-of-arrays layout below.  Every kernel receives a DevState by
// value: the carved pointers, the handle's constants and the current step's
// input/output pointers.
#pragma once

#include <cstddef>
#include <cstdint>

#include <cuda_runtime.h>

#include "prefixshield.h"

namespace ps {

// ---- constants -------------------------------------------------------------
constexpr uint32_t kNone = 0xFFFFFFFFu;           // empty slot / no block
constexpr int kProb = 0, kNormal = 1, kReuse = 2;  // retention classes (Eq. 9 order)
constexpr uint64_t kMaxPos = (1ull << 18) - 1;   // full blocks per request
constexpr uint64_t kMaxStep = (1ull << 31) - 1;  // steps (step tags keep 32 bits)
constexpr int kTableWays = 8;    // native prefix table: 8 x 16 B entries per 128 B bucket
constexpr int kClaimWays = 4;    // per-step claim map: 4 x 32 B entries per bucket
constexpr int kRadixBits = 8;
constexpr int kRadixBins = 1 << kRadixBits;
constexpr int kSegBlocks = 32;   // blocks of one chunk half (a warp's width)
constexpr int kChunkBlocks = 2 * kSegBlocks;  // blocks of one prompt hashed by one warp (a chunk)
constexpr int kBmChunk = 256;    // bitmap words per CTA of the id-list compaction
constexpr int kValTile = 256;    // requests per CTA of the input validation (one published total each)
constexpr uint64_t kP61 = (1ull << 61) - 1;  // chain modulus, a Mersenne prime

// Recency stamp (native free-queue order): larger = more recently released.
// One running counter over the steps: request i's block m gets
// base + (full blocks of the step's earlier requests) + (n_i - 1 - m), so a
// request's deeper blocks (released first) are older.
__host__ __device__ __forceinline__ uint64_t make_stamp(uint64_t base, uint64_t pbase, uint64_t n, uint64_t m) {
  return base + pbase + (n - 1 - m);
}

// ---- table entries ---------------------------------------------------------
struct __align__(16) TableEntry {   // native prefix table (group, key) -> block
  uint64_t key;
  uint32_t blk;   // kNone when the slot is empty
  uint32_t grp;
};

struct __align__(32) ClaimEntry {   // per-step: first request that needs a new key
  uint64_t key;     // 0 when empty
  uint32_t minreq;  // lowest request index containing the key (atomicMin)
  uint32_t tcnt;    // in-step touches
  uint32_t promo;   // lowest request index whose touch promotes it
  uint32_t pad;
  uint64_t stamp;   // recency stamp of the latest in-step touch (atomicMax; 0: none)
};
__host__ __device__ __forceinline__ ClaimEntry empty_claim() {
  ClaimEntry e{};
  e.key = 0; e.minreq = kNone; e.tcnt = 0; e.promo = kNone; e.pad = 0; e.stamp = 0;
  return e;
}

struct __align__(32) HistEntry {    // (group, prefix id) -> reference history
  uint64_t p;       // 0 when empty
  uint32_t g1;      // group + 1
  uint32_t refadm;  // reference count (bits 0..30) | admitted (bit 31)
  uint64_t ftag;    // (step << 32) | ~first request of the step with this entry
  uint64_t atag;    // (step << 32) | ~first request of the step that admitted
};

// Device-resident control block: persistent scalars and per-step scalars.
struct Ctl {
  // persistent
  int32_t sticky;          // PS_OK or PS_ERR_CAPACITY
  int32_t pad0;
  uint64_t step;           // index of the step being / next to be processed (from 1)
  uint64_t stamp_base;     // first recency stamp of this step (from 1)
  int64_t t_prev;          // last refill time
  int64_t n_resident;
  int64_t hist_live;
  uint64_t s3_ctr, ghost_ctr;
  int64_t s3_nS, s3_nM;             // queue sizes (pinned members included)
  int64_t s3_len[2];                // small (0) and main (1) queue arrays: entries, oldest first
  int32_t s3_buf;                   // which of the two array buffers holds the queues
  int32_t ghost_rbuf;               // which of the two ghost rings holds the FIFO
  uint64_t ghost_head, ghost_tail;  // ghost FIFO window [tail, head) (absolute positions)
  int64_t ghost_live;               // live ghost entries
  // per step
  int32_t status;          // this step's status
  int32_t pad1;
  int64_t T, nblocks, nsegs;
  int64_t pinned, n_inval, total_claims, avail, need, nfree, ftake, mvict;
  int64_t hist_new;
  int64_t n_evicted, n_alloc, n_victims_marked;
  int64_t m_fb;            // prefixshield: victims left to the global fallback
  int32_t sel_ntie, sel_k; // prefixshield tie bookkeeping
  int64_t lst_n;              // members of the select's split list
  uint32_t ticket;         // last-block-done counter for the radix passes and the split
  int32_t nlaunch;         // kernels launched by the step (conditional bodies run or not)
  int32_t wide_nrows;      // segments counted by the last first-digit pass
  int32_t internal_error;  // an invariant of the step failed (reported, never expected)
  // indexed queues (PS_FLAG_INDEXED_QUEUES)
  int32_t lg_buf;          // entry buffer holding the logs (0 or 1)
  int32_t lg_ntk;          // takes of the select phase in progress
  int32_t lg_nchunks;      // chunks of the scan in progress
  int32_t lg_more;         // a take's window ended short of its last victim: another round
  int32_t lg_cmp;          // a log lacks room for this step's appends: compact first
  uint32_t lg_ticket;      // last-CTA-done counter of the append and compaction writes
  uint32_t hash_ticket;    // chunks handed out to k_hash_lookup's CTAs, in order
  uint32_t v_ticket;       // k_validate: CTAs done (the last one finishes the call)
  uint32_t v_bad;          // k_validate: bit 0 an invalid request, bit 1 a look-back ran out
  uint64_t v_sum;          // k_validate: blocks (high half) and chunks (low half) of the call
};

// One hashing chunk: up to kChunkBlocks consecutive blocks of one request.
struct __align__(16) ChunkDesc {
  int64_t o0;      // the request's first token
  uint32_t req;    // request index
  int32_t n;       // the request's full blocks
  int32_t pbase;   // position of the request's block 0
  int32_t k;       // this chunk's index within the request
  uint32_t group;  // the request's group
  int32_t sb;      // the request's first chunk
};

// Per-segment state of the segmented radix select.
struct __align__(16) SelSeg {
  uint64_t prefix;   // key bits fixed so far
  uint64_t mask;     // which bits are fixed
  int64_t rank;      // 1-based rank still to locate inside the prefix class
  int32_t active;    // 1 while this segment selects
  int32_t incl;      // 1: victims are keys <= prefix; 0: keys < prefix
  uint64_t kmin, kmax;  // a range holding every candidate key of the segment
  uint64_t qmin, qmax;  // range of the segment's keys on the split list
};

// Candidates of one (segment, retention class): their number and the ranges
// of their stamps' top and bottom 32 bits.
struct ClsRange {
  uint32_t cnt, hmin, hmax, lmin, lmax;
};

// ---- indexed queues (the per-group, per-segment queues of Sec. VIII) -------
// Each queue is a log of (block, stamp) entries in stamp order: a block is
// appended at the end of every step that restamps or admits it, and an entry
// is live while the block is resident with that stamp.  Logs 3g + k hold
// group g's blocks of class k; logs 3G + k hold every group's blocks of
// class k (class 0 only, for all classes, when the policy ignores classes).
constexpr int kLogChunk = 1024;  // log entries per chunk of a scan
constexpr int kAppChunk = 256;   // stamps per chunk of the end-of-step append
constexpr int kMaxLogs = PS_MAX_GROUPS * 3 + 3;
struct LogDesc {
  int64_t start, head, tail, end;  // positions in the current entry buffer
};
// One log's share of a select phase: consume its first 'want' live entries.
struct LogTake {
  int64_t want;  // live entries to consume (with 'tie', the last one is recorded, not taken)
  int64_t got;   // consumed in earlier rounds
  int64_t cur;   // where this round's window starts
  int64_t wend;  // where it ends
  int32_t log;
  int32_t tie;   // the last entry is the group's tie candidate (Eq. 7)
  int32_t done;  // the last entry was found (this round or earlier)
  int32_t pad;
};
struct TieItem {
  uint64_t key;  // (class, stamp) order key of the tied group's next candidate
  int64_t pos;   // its position in the log
  uint32_t blk;
  int32_t log;
};
constexpr int kClasses = 3;
// The first digit of a select is 16 bits wide while at most kWideRows
// segments count (8 bits otherwise).
constexpr int kWideRows = 64;
constexpr int kWideBins = 1 << 16;

// ---- S3-FIFO as sequence-ordered arrays ------------------------------------
// Both queues are arrays of block ids in sequence order (oldest first),
// rebuilt every step from the step's closed-form plan; chunks of kS3Chunk
// entries are the unit of the per-step passes.
constexpr int kS3Chunk = 2048;
constexpr int kS3Bins = 16;      // frequencies 0..15 (a larger cap takes the sequential kernel)
struct S3Chunk {
  uint32_t nlive, nu, nev, pad;  // live entries, unpinned ones, unpinned with f < move threshold
  uint32_t hist[kS3Bins];        // unpinned entries by frequency
};
struct S3Base {                  // exclusive prefixes of a chunk (per-region or main-then-small order)
  uint32_t u, ev, mv, keep, ge, gt, pad0, pad1;
};
struct S3Plan {
  int64_t lenS, lenM;    // queue arrays at step start
  int64_t pcut;          // unpinned small entries before this array position are consumed
  int64_t kS;            // small-queue evictions (ghost pushes)
  int64_t MA;            // small -> main moves
  int64_t UMo;           // unpinned main entries (the main phase's visit list starts with them)
  int64_t nL;            // main phase's visit list: UMo, then the moved blocks
  int64_t P;             // visit-list index of the final round's last visit (-1: no main phase)
  int64_t rge_P1, rgt_P1;  // visit-list entries at or before P with f >= Rs / f > Rs
  int64_t base_Rm1, base_R;  // reinsertions in rounds before Rs - 1 / before Rs
  int64_t nG1, nUnvMov, nMid;
  int64_t nKeepS, nKeepM;
  uint64_t ctr0, ctr_end;
  int32_t Rs;            // the final round of the main phase (0 without one)
  int32_t fb;            // 1: the sequential kernel takes the step
  int32_t gc;            // 1: the ghost FIFO is compacted into the other ring
  int32_t rbuf;          // ring holding the window at step start
  uint64_t g_head, g_tail, ra0;  // window at step start; first ring chunk's start
  int64_t nrch;          // ring chunks over the window
  int64_t live_old;      // live ghost entries at step start
  int64_t X;             // oldest live entries the pushes trim (may exceed live_old)
  int64_t born;          // pushes trimmed at once: max(0, X - live_old)
  uint64_t pbase;        // push t (t >= born) goes to position pbase + t
  uint64_t q;            // new window start without compaction
  uint64_t gctr0;        // ghost counter at step start
  int64_t n_ins, hits;   // inserted blocks; ghost hits among them
};

// Per-call arguments of a step or probe, in device memory: the step's kernels
// read them at entry, so one captured CUDA graph serves every step.
struct StepArgs {
  int64_t now;
  int32_t R;
  int32_t tokens_aligned16;
  const int32_t* in_group;
  const int64_t* in_offsets;
  const int32_t* in_tokens;
  const int32_t* in_contract;
  const uint64_t* in_prefix;
  ps_step_out_t out;
};

struct DevState {
  // constants
  int64_t N;
  int32_t bs, G, C, policy;
  uint32_t flags;
  int32_t fp_shift;
  int64_t eps;
  uint64_t hash_seed;
  uint64_t chain_mul, digest_mul;  // Kc, Kd of the key chain (mod 2^61-1)
  int64_t max_segments;
  int64_t rho[PS_MAX_CONTRACTS], beta[PS_MAX_CONTRACTS];
  int64_t rho_min;
  int32_t s3_small_pct, s3_freq_cap, s3_move_min;
  int64_t s3_small_cap, s3_ghost_cap;
  uint32_t gh_nbuckets_log2;
  uint64_t ghost_ring_cap;  // power of two
  int32_t max_requests;
  int64_t max_tokens, max_blocks;
  int64_t history_capacity;
  uint32_t tb_nbuckets_log2, cl_nbuckets_log2, hist_cap_log2;
  int64_t nwords;          // resident bitmap words
  // persistent state
  Ctl* ctl;
  uint64_t* blk_key;
  uint64_t* blk_stamp;
  uint64_t* blk_prefix;
  uint64_t* blk_promo;     // (step << 32) | ~promoting request (atomicMax)
  uint64_t* blk_s3seq;
  uint16_t* blk_group;
  uint8_t* blk_contract;
  uint8_t* blk_klass;
  uint8_t* blk_flags;      // bit0 resident, bit1 S3-FIFO main queue
  uint32_t* blk_freq;      // S3-FIFO counter, unclamped (read as min(cap, f))
  uint32_t* blk_acc;
  uint32_t* blk_slot;      // table slot of a resident block
  uint32_t* blk_pin;       // step tag: hit in this step
  uint32_t* blk_inval;     // step tag: invalidated in this step
  uint32_t* res_bits;      // resident bitmap
  // S3-FIFO queues: per buffer, the small queue's ids then the main queue's,
  // each in a region of s3_np entries, oldest first (sequence order)
  int64_t s3_np;           // region stride: N rounded up to a whole chunk
  int64_t s3_nch;          // chunks a region can hold
  int64_t s3_nrch;         // chunks a ghost ring can hold (plus one)
  uint32_t* s3_arr;        // [2][2][s3_np]
  TableEntry* ghost_map;   // (group, key) -> ring index (in blk)
  uint32_t* ghost_ovf;
  uint64_t* ghost_sq;      // per map slot: the entry's ghost sequence number
  uint32_t* ghost_ring;    // [2][ghost_ring_cap] map slot of each FIFO position
  uint32_t* ghost_bits;    // [2][ghost_ring_cap / 32] live FIFO positions
  TableEntry* table;
  uint32_t* table_ovf;     // per bucket: live keys probing past it
  int64_t* ledger;         // B_{g,c}, fixed point
  int64_t* ledger_b0;      // per step: B_{g,c} refilled to now, before the step's charges
  int32_t* contract_of_group;
  uint32_t* key_words;     // NH key schedule, bs + 2 words
  uint64_t* kc_pow;        // Kc^k mod p, k = 0..kSegBlocks, then Kc^(kChunkBlocks t), t = 0..kSegBlocks
  int64_t* stats;          // [G][PS_NUM_STATS]
  HistEntry* hist;
  // per-step scratch
  int32_t* rq_n;           // full blocks
  int32_t* rq_pbase;       // first position index of the request
  int32_t* rq_h;           // cached prefix length
  int32_t* rq_s;           // first own claim
  int32_t* rq_cbase;       // exclusive scan of claims
  int32_t* rq_a;           // granted (admitted) blocks
  int32_t* rq_e;           // in-step hits
  uint32_t* rq_fu;         // first ungranted in-step position
  int32_t* rq_cid;         // contract
  uint32_t* rq_hs;         // history slot
  uint64_t* rq_p;          // prefix id
  uint8_t* rq_flags;       // bit0 proven, bit1 gate open
  uint8_t* rq_knew;        // class of newly admitted blocks
  uint64_t* pos_key;       // chain partial, then the block key
  uint32_t* pos_req;       // request of the position
  uint32_t* pos_m;         // the position's block index within its request
  ChunkDesc* chunks;       // hashing chunks of the call, in request order
  uint64_t* val_tile;      // k_validate's published per-tile totals (zero between calls)
  uint64_t* seg_word;      // the chunk's published chain total and miss bit (k_hash_lookup)
  uint32_t* pos_blk;       // resident block hit by lookup (or kNone)
  uint32_t* pos_claim;     // claim-map slot (or kNone)
  uint8_t* pos_elig;       // touch was promotion-eligible
  ClaimEntry* claims;
  uint32_t* bm_victim;     // per-step bitmaps over block ids
  uint32_t* bm_inval;
  uint64_t* csk;           // candidate sort keys (~0 = not a candidate)
  int64_t* grp_qsize;      // candidates per group
  int64_t* grp_P;          // projected score P^(0)_g = normalized debt
  int64_t* grp_delta;      // Eq. 8 decrement
  int64_t* grp_x;          // victims taken from the group in the debt phase (StaticQuota: its overflow)
  int64_t* grp_pinned;     // blocks pinned this step, per group (StaticQuota grants)
  uint8_t* grp_full;       // the debt phase takes all of the group's candidates
  SelSeg* sel;             // [G] segments
  ClsRange* cls;           // [G * kClasses] candidates per (segment, class)
  uint32_t* hist_bins;     // [G][256] radix histogram
  uint32_t* wide_bins;     // [kWideRows][65536] first-digit histograms (or [G][256])
  uint32_t* wide_coarse;   // [kWideRows][256] the 16-bit histograms summed by their top byte
  int16_t* wide_seg;       // [G] segment of each first-digit row
  uint64_t* lst_key;       // split list of the select: key, block, segment
  uint32_t* lst_blk;
  uint16_t* lst_seg;
  int32_t* bm_chunk_cnt;   // [3][chunks] bitmap compaction counts
  // S3-FIFO per-step scratch
  uint8_t* s3_attr;        // [2][s3_np] per queue entry: bit0 live, bit1 unpinned, bits 4-7 frequency
  S3Chunk* s3_ck;          // [2][s3_nch] per-chunk counts
  S3Base* s3_base;         // [2][s3_nch] per-chunk exclusive bases
  uint32_t* s3_rck;        // [s3_nrch] live ghost entries per ring chunk of the window
  uint32_t* s3_rbase;      // [s3_nrch] their exclusive prefix
  S3Plan* s3_plan;
  uint8_t* s3_hit;         // [max_blocks] inserted block found in the ghost
  uint32_t* s3_ick;        // [max_blocks / kS3Chunk + 1] ghost hits per chunk of inserts
  // indexed queues (allocated only with PS_FLAG_INDEXED_QUEUES)
  int32_t lg_on;           // victims come from the queues instead of a candidate scan
  int32_t lg_L;            // logs: 3G + 3
  int64_t lg_P;            // entries per buffer
  int64_t lg_max_chunks;   // chunks a scan can span
  int64_t lg_app_chunks;   // append chunks of the largest step
  uint32_t* lg_blk;        // [2][P] entries: block
  uint64_t* lg_st;         // [2][P]          stamp when appended
  LogDesc* lg_desc;        // [L]
  LogDesc* lg_new;         // [L] layout after a compaction
  int64_t* lg_live;        // [L] live entries (candidates)
  int64_t* lg_add;         // [L] entries this step appends
  int64_t* lg_pin;         // [L] entries this step's pins take out (applied once the step goes ahead)
  uint32_t* lg_slot;       // [max_blocks] block holding each stamp of this step
  uint32_t* lg_app;        // [L][app_chunks] append counts per chunk, then offsets
  LogTake* lg_tk;          // [L] takes of a select phase
  int32_t* lg_c0;          // [L + 1] first chunk of each take (or log)
  uint32_t* lg_ck;         // [max_chunks] live entries per chunk (compaction)
  int64_t* lg_ck_out;      // [max_chunks] a take round's look-back status words; in a
                           // compaction, where each chunk's live entries go
  TieItem* lg_tie;         // [G]
  StepArgs* args;          // this call's arguments (device memory)
  // current step inputs / outputs (kernels refresh them from *args)
  int64_t now;
  int32_t R;
  const int32_t* in_group;
  const int64_t* in_offsets;
  const int32_t* in_tokens;
  const int32_t* in_contract;
  const uint64_t* in_prefix;
  int32_t tokens_aligned16;
  ps_step_out_t out;
};

// ---- hashing (published definitions, implemented here independently) -----
// SplitMix64 output function (Steele, Lea, Flood 2014), used as a mixer.
__host__ __device__ __forceinline__ uint64_t mix64(uint64_t z) {
  z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
  z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
  return z ^ (z >> 31);
}
__host__ __device__ __forceinline__ uint64_t fix_reserved(uint64_t h) {
  return (h == 0 || h == ~0ull) ? 1ull : h;
}
__host__ __device__ __forceinline__ uint64_t chain_seed(uint64_t seed, int32_t g) {
  return mix64(seed ^ ((uint64_t)(g + 1) * 0x9E3779B97F4A7C15ull));
}
__device__ __forceinline__ uint32_t table_home(uint64_t key, uint32_t g, uint32_t log2nb) {
  uint64_t x = (key ^ ((uint64_t)(g + 1) * 0x9E3779B97F4A7C15ull)) * 0xD6E8FEB86659FD93ull;
  return (uint32_t)(x >> (64 - log2nb));
}
__device__ __forceinline__ uint32_t claim_home(uint64_t key, uint32_t log2nb) {
  return (uint32_t)((key * 0xC2B2AE3D27D4EB4Full) >> (64 - log2nb));
}
__device__ __forceinline__ uint32_t hist_home(uint64_t p, uint32_t g, uint32_t log2cap) {
  uint64_t x = (p ^ ((uint64_t)(g + 1) * 0xFF51AFD7ED558CCDull)) * 0x9E3779B97F4A7C15ull;
  return (uint32_t)(x >> (64 - log2cap));
}

// ---- host launchers (ps_kernels.cu) ----------------------------------------
// Optional stage events (profiling hook) and the launch count of a step.
struct StepTrace {
  cudaEvent_t ev[PS_NUM_STAGES + 1];
  bool timing = false;
  int launches = 0;
};

// Stream capture of a step: a second private stream on which the bodies of
// conditional graph nodes are captured (phases that many steps skip).
struct CaptureCtx {
  cudaStream_t aux;   // bodies of top-level conditional nodes
  cudaStream_t aux2;  // bodies of conditional nodes inside those
  cudaStream_t side;  // a parallel branch of the step graph (the candidate scan)
  cudaEvent_t fork, join;
  cudaStream_t side2;  // a second branch (in-step hits, metering, touch passes)
  cudaEvent_t fork2, join2;
};

// Copy the call's arguments from device memory into the kernel's DevState,
// then wait for the preceding kernel of the step.  Step kernels are launched
// with programmatic stream serialization, so a kernel's CTAs may already be
// resident while its predecessor runs: every kernel passes this wait before it
// reads or writes any state, and then lets its own successor be scheduled.
// The argument block itself is written only by the host before the step.
// Without that launch attribute both instructions are no-ops.
__device__ __forceinline__ DevState with_args(DevState s) {
  const StepArgs* a = s.args;
  if (a != nullptr) {
    s.now = a->now;
    s.R = a->R;
    s.tokens_aligned16 = a->tokens_aligned16;
    s.in_group = a->in_group;
    s.in_offsets = a->in_offsets;
    s.in_tokens = a->in_tokens;
    s.in_contract = a->in_contract;
    s.in_prefix = a->in_prefix;
    s.out = a->out;
  }
  asm volatile("griddepcontrol.wait;" ::: "memory");
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
  if (a != nullptr && blockIdx.x == 0 && threadIdx.x == 0) atomicAdd(&s.ctl->nlaunch, 1);
  return s;
}
// The host-side argument block of a DevState.
inline StepArgs args_of(const DevState& s) {
  StepArgs a{};
  a.now = s.now; a.R = s.R; a.tokens_aligned16 = s.tokens_aligned16;
  a.in_group = s.in_group; a.in_offsets = s.in_offsets; a.in_tokens = s.in_tokens;
  a.in_contract = s.in_contract; a.in_prefix = s.in_prefix; a.out = s.out;
  return a;
}
// Kernel attributes (shared-memory opt-ins), set once per process before
// any launch or capture.
void configure_kernels(const DevState& s);
void launch_init(const DevState& s, cudaStream_t st);
int32_t launch_step(const DevState& s, cudaStream_t st, StepTrace* tr, const CaptureCtx* cap = nullptr);
// Indexed queues (ps_queues.cu).  The select phases are 0 Alg. 2's debt
// phase, 1 its global fallback, 2 lru, 3 StaticQuota.
void launch_queue_init(const DevState& s, cudaStream_t st);
int32_t launch_queue_cand(const DevState& s, cudaStream_t st, int* launches);
int32_t launch_queue_select(const DevState& s, cudaStream_t st, const CaptureCtx* cap, int phase, int depth,
                            bool plain_first, int* launches);
int32_t launch_queue_append(const DevState& s, cudaStream_t st, const CaptureCtx* cap, int* launches);
// S3-FIFO (ps_s3fifo.cu)
// The select: per-chunk counts, the closed-form plan, the sequential kernel
// (used when the plan does not apply), the plan's application.
// plain_first: the first kernel follows a fork of the step graph (a plain
// launch: a programmatic edge is kept for a kernel's only dependent).
int32_t launch_s3_select(const DevState& s, cudaStream_t st, bool plain_first, int* launches);
// After the insertions: ghost lookups of the new blocks, their array places.
int32_t launch_s3_insert(const DevState& s, cudaStream_t st, int* launches);
// A step's outputs (device) written into page-locked host buffers, the id
// lists by their device-side counts (ps_step_host_async).
void launch_host_out(const ps_step_out_t& dev, const ps_step_out_t& host, int32_t R, int32_t G, cudaStream_t st);
// Read-only cached-prefix probe; 'out' receives h_i per request, 'status' the outcome.
int32_t launch_probe(const DevState& s, cudaStream_t st, int32_t* out, int32_t* status);

}  // namespace ps
