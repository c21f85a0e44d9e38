// C ABI of the prefix-cache step library (declared in include/prefixshield.h).
//
// Host side only: argument checks, the workspace layout, the handle, and the
// copies of the test hooks.  Every stage of a step runs in the kernels of
// ps_kernels.cu.
#include <cstdlib>
#include <cstring>
#include <new>
#include <vector>

#include "ps_internal.cuh"

using namespace ps;

struct ps_handle {
  DevState base;        // constants and carved pointers; per-step fields unused
  void* workspace;
  size_t workspace_bytes;
  int device;
  // staging areas for ps_step_host() (slot 0) and ps_step_host_async() (slots 0, 1)
  struct Staging {
    int32_t* group;
    int64_t* offsets;
    int32_t* tokens;
    int32_t* contract;
    uint64_t* prefix;
  } stg[2];
  ps_step_out_t st_out;
  cudaStream_t copy_stream = nullptr;  // the pipelined inputs' copies
  cudaEvent_t in_ready[2] = {nullptr, nullptr}, slot_free[2] = {nullptr, nullptr}, done[2] = {nullptr, nullptr};
  const ps_host_out_t* pending[2] = {nullptr, nullptr};
  StepTrace trace;
  std::vector<int32_t> contract_of_group;
  // the step as one CUDA graph, captured on a private stream at first use
  StepArgs* step_args;
  cudaStream_t cap_stream = nullptr;
  cudaStream_t cap_aux = nullptr;   // conditional bodies are captured here
  cudaStream_t cap_aux2 = nullptr;  // and bodies nested in them here
  cudaStream_t cap_side = nullptr;  // a parallel branch of the step graph
  cudaStream_t cap_side2 = nullptr; // a second one
  cudaEvent_t cap_fork = nullptr, cap_join = nullptr, cap_fork2 = nullptr, cap_join2 = nullptr;
  cudaGraph_t graph = nullptr;
  cudaGraphExec_t exec = nullptr;
  bool exec_timing = false;
  bool use_graph = true;
};

namespace {

inline size_t align_up(size_t x, size_t a) { return (x + a - 1) / a * a; }
inline uint32_t log2_pow2_at_least(uint64_t v) {
  uint32_t l = 0;
  while ((1ull << l) < v) ++l;
  return l;
}

// SplitMix64 stream (Steele, Lea, Flood 2014) for the key schedule.
uint64_t splitmix_next(uint64_t* st) {
  *st += 0x9E3779B97F4A7C15ull;
  return mix64(*st);
}
uint64_t host_mul61(uint64_t a, uint64_t b) { return (uint64_t)(((unsigned __int128)a * b) % kP61); }

// Key schedule: bs + 2 NH words, then the chain and digest multipliers.
struct KeySchedule {
  std::vector<uint32_t> words;
  uint64_t kc, kd;
  std::vector<uint64_t> kc_pow;
};
KeySchedule key_schedule(uint64_t seed, int32_t bs) {
  KeySchedule k;
  uint64_t st = seed;
  k.words.resize((size_t)bs + 2);
  for (auto& w : k.words) w = (uint32_t)splitmix_next(&st);
  k.kc = splitmix_next(&st) % kP61;
  k.kd = splitmix_next(&st) % kP61;
  if (k.kc == 0) k.kc = 1;
  if (k.kd == 0) k.kd = 1;
  // Kc^j for j = 0..kSegBlocks
  k.kc_pow.resize(2 * (kSegBlocks + 1));
  k.kc_pow[0] = 1;
  for (int j = 1; j <= kSegBlocks; ++j) k.kc_pow[j] = host_mul61(k.kc_pow[j - 1], k.kc);
  // then the powers of Kc^kChunkBlocks (one chunk's multiplier), t = 0..kSegBlocks
  const uint64_t kc_chunk = host_mul61(k.kc_pow[kSegBlocks], k.kc_pow[kSegBlocks]);
  k.kc_pow[kSegBlocks + 1] = 1;
  for (int t = 1; t <= kSegBlocks; ++t) k.kc_pow[kSegBlocks + 1 + t] = host_mul61(k.kc_pow[kSegBlocks + t], kc_chunk);
  return k;
}

int32_t upload_constants(ps_handle* h, cudaStream_t st) {
  const KeySchedule ks = key_schedule(h->base.hash_seed, h->base.bs);
  if (cudaMemcpyAsync(h->base.key_words, ks.words.data(), ks.words.size() * 4, cudaMemcpyHostToDevice, st) !=
          cudaSuccess ||
      cudaMemcpyAsync(h->base.kc_pow, ks.kc_pow.data(), ks.kc_pow.size() * 8, cudaMemcpyHostToDevice, st) !=
          cudaSuccess ||
      cudaMemcpyAsync(h->base.contract_of_group, h->contract_of_group.data(), h->contract_of_group.size() * 4,
                      cudaMemcpyHostToDevice, st) != cudaSuccess ||
      cudaStreamSynchronize(st) != cudaSuccess)
    return PS_ERR_CUDA;
  return PS_OK;
}

int32_t check_params(int64_t N, int32_t bs, int32_t G, int32_t policy, const ps_params_t* P) {
  if (!P || N <= 0 || N > (1ll << 30)) return PS_ERR_INVALID_ARG;
  if (bs != 2 && bs != 4 && bs != 8 && bs != 16 && bs != 32 && bs != 64) return PS_ERR_INVALID_ARG;
  if (G <= 0 || G > PS_MAX_GROUPS || policy < 0 || policy > 3) return PS_ERR_INVALID_ARG;
  if (P->num_contracts < 1 || P->num_contracts > PS_MAX_CONTRACTS) return PS_ERR_INVALID_ARG;
  if (P->fp_shift < 0 || P->fp_shift > 30 || P->epsilon_fp < 0) return PS_ERR_INVALID_ARG;
  int64_t rmin = P->rho_fp[0], rmax = P->rho_fp[0];
  for (int c = 0; c < P->num_contracts; ++c) {
    if (P->rho_fp[c] <= 0 || P->beta_fp[c] < 0) return PS_ERR_INVALID_ARG;
    if (P->beta_fp[c] > (1ll << 52) || P->rho_fp[c] > (1ll << 52)) return PS_ERR_INVALID_ARG;
    if (P->rho_fp[c] < rmin) rmin = P->rho_fp[c];
    if (P->rho_fp[c] > rmax) rmax = P->rho_fp[c];
  }
  // Eq. 8's decrement rho_min/rho_max in fixed point must be at least 1.
  if ((int64_t)(((__int128)1 << P->fp_shift) * rmin / rmax) < 1) return PS_ERR_INVALID_ARG;
  for (int g = 0; g < G; ++g)
    if (P->contract_of_group[g] < 0 || P->contract_of_group[g] >= P->num_contracts) return PS_ERR_INVALID_ARG;
  if (P->s3_small_pct < 1 || P->s3_small_pct > 100 || P->s3_freq_cap < 1 || P->s3_freq_cap > 255)
    return PS_ERR_INVALID_ARG;
  if (P->s3_move_min_freq < 1 || P->history_capacity < 1 || P->history_capacity > (1ll << 28))
    return PS_ERR_INVALID_ARG;
  return PS_OK;
}

// Workspace carving.  One pass computes offsets (base == nullptr) or
// assigns pointers; every region starts on a 256-byte boundary.
struct Carver {
  char* base;
  size_t off = 0;
  template <typename T>
  T* take(size_t count) {
    off = align_up(off, 256);
    T* p = base ? reinterpret_cast<T*>(base + off) : nullptr;
    off += sizeof(T) * (count ? count : 1);
    return p;
  }
};

struct Dims {
  int64_t N, max_tokens, max_blocks, nwords, hist_cap, max_segments;
  int64_t s3_small_cap, s3_ghost_cap;
  uint64_t ghost_ring_cap;
  int64_t s3_np, s3_nch, s3_nrch;
  uint32_t gh_log2;
  int32_t bs, G, C, max_requests;
  uint32_t tb_log2, cl_log2, hist_log2;
  // indexed queues
  bool lg;
  int32_t lg_L;
  int64_t lg_P, lg_max_chunks, lg_app_chunks;
};

Dims make_dims(int64_t N, int32_t bs, int32_t G, const ps_params_t* P, int32_t max_requests, int64_t max_tokens) {
  Dims d{};
  d.N = N; d.bs = bs; d.G = G; d.C = P->num_contracts; d.max_requests = max_requests;
  d.max_tokens = max_tokens;
  d.max_blocks = max_tokens / bs;
  d.max_segments = d.max_blocks / kChunkBlocks + max_requests + 1;
  d.nwords = (N + 31) / 32;
  // native table: 8-way buckets at load <= 1/2
  // 8-way buckets for 4N entries: at most a quarter full, so a probe rarely
  // continues past its home bucket
  d.tb_log2 = log2_pow2_at_least((uint64_t)((N + 1) / 2 > 1 ? (N + 1) / 2 : 1));
  if (d.tb_log2 < 1) d.tb_log2 = 1;
  // claim map: 4-way buckets, at least one slot per block of a step (load <=
  // 1 even if every block of a full step is new; about a quarter of that in
  // typical steps)
  d.cl_log2 = log2_pow2_at_least((uint64_t)(d.max_blocks / 4 > 1 ? d.max_blocks / 4 : 1));
  if (d.cl_log2 < 1) d.cl_log2 = 1;
  d.hist_log2 = log2_pow2_at_least((uint64_t)(2 * (P->history_capacity + max_requests)));
  if (d.hist_log2 < 1) d.hist_log2 = 1;
  d.hist_cap = P->history_capacity;
  // S3-FIFO: small queue max(1, floor(N * pct / 100)); ghost holds the rest
  d.s3_small_cap = N * P->s3_small_pct / 100 > 1 ? N * P->s3_small_pct / 100 : 1;
  d.s3_ghost_cap = N - d.s3_small_cap;
  d.gh_log2 = log2_pow2_at_least((uint64_t)((d.s3_ghost_cap + 3) / 4 > 1 ? (d.s3_ghost_cap + 3) / 4 : 1));
  if (d.gh_log2 < 1) d.gh_log2 = 1;
  // S3-FIFO queue arrays: a region of N entries rounded up to whole chunks.
  // Ghost FIFO ring: room for twice the ghost's capacity plus a step's pushes
  // (at most max_blocks), so compactions are rare; at least two chunks.
  d.s3_np = (N + kS3Chunk - 1) / kS3Chunk * kS3Chunk;
  d.s3_nch = d.s3_np / kS3Chunk;
  // At most 2^31 positions: a FIFO index must stay below the map's empty
  // marker (0xFFFFFFFF), and 2^31 still holds a full ghost (< 2^30 entries)
  // plus a step's pushes (< 2^30) after a compaction.
  {
    const uint64_t want = (uint64_t)(2 * (d.s3_ghost_cap + d.max_blocks));
    d.ghost_ring_cap = 1ull << log2_pow2_at_least(want > 2 * (uint64_t)kS3Chunk ? want : 2 * (uint64_t)kS3Chunk);
    if (d.ghost_ring_cap > (1ull << 31)) d.ghost_ring_cap = 1ull << 31;
  }
  d.s3_nrch = (int64_t)(d.ghost_ring_cap / kS3Chunk) + 1;
  // indexed queues: at most two live entries a block (its group's log and its
  // class's global log) and two a position of a step; each buffer holds eight
  // times that, so a compaction leaves at least seven eighths free
  d.lg = (P->flags & PS_FLAG_INDEXED_QUEUES) != 0;
  d.lg_L = G * kClasses + kClasses;
  d.lg_P = 2 * 8 * (N + d.max_blocks);
  d.lg_max_chunks = d.lg_P / kLogChunk + d.lg_L + 2;
  d.lg_app_chunks = (d.max_blocks + kAppChunk - 1) / kAppChunk;
  if (d.lg_app_chunks < 1) d.lg_app_chunks = 1;
  return d;
}

// Returns the total size; fills s / h pointers when base != nullptr.
size_t carve(const Dims& d, char* base, DevState* s, ps_handle* h) {
  Carver cv{base};
  const size_t N = (size_t)d.N, R = (size_t)d.max_requests, B = (size_t)d.max_blocks, G = (size_t)d.G;
  DevState t{};
  t.ctl = cv.take<Ctl>(1);
  t.blk_key = cv.take<uint64_t>(N);
  t.blk_stamp = cv.take<uint64_t>(N);
  t.blk_prefix = cv.take<uint64_t>(N);
  t.blk_promo = cv.take<uint64_t>(N);
  t.blk_s3seq = cv.take<uint64_t>(N);
  t.blk_group = cv.take<uint16_t>(N);
  t.blk_contract = cv.take<uint8_t>(N);
  t.blk_klass = cv.take<uint8_t>(N);
  t.blk_flags = cv.take<uint8_t>(N);
  t.blk_freq = cv.take<uint32_t>(N);
  t.blk_acc = cv.take<uint32_t>(N);
  t.blk_slot = cv.take<uint32_t>(N);
  t.blk_pin = cv.take<uint32_t>(N);
  t.blk_inval = cv.take<uint32_t>(N);
  const size_t zero_end = cv.off;  // everything above starts zeroed
  t.res_bits = cv.take<uint32_t>((size_t)d.nwords);
  t.s3_arr = cv.take<uint32_t>(4 * (size_t)d.s3_np);
  t.ghost_map = cv.take<TableEntry>((size_t)kTableWays << d.gh_log2);
  t.ghost_ovf = cv.take<uint32_t>((size_t)1 << d.gh_log2);
  t.ghost_sq = cv.take<uint64_t>((size_t)kTableWays << d.gh_log2);
  t.ghost_ring = cv.take<uint32_t>(2 * (size_t)d.ghost_ring_cap);
  t.ghost_bits = cv.take<uint32_t>(2 * (size_t)(d.ghost_ring_cap / 32));
  t.table = cv.take<TableEntry>((size_t)kTableWays << d.tb_log2);
  t.table_ovf = cv.take<uint32_t>((size_t)1 << d.tb_log2);
  t.ledger = cv.take<int64_t>(G * d.C);
  t.ledger_b0 = cv.take<int64_t>(G * d.C);
  t.contract_of_group = cv.take<int32_t>(G);
  t.key_words = cv.take<uint32_t>((size_t)d.bs + 2);
  t.kc_pow = cv.take<uint64_t>(2 * ((size_t)kSegBlocks + 1));
  t.stats = cv.take<int64_t>(G * PS_NUM_STATS);
  t.hist = cv.take<HistEntry>((size_t)1 << d.hist_log2);
  t.rq_n = cv.take<int32_t>(R);
  t.rq_pbase = cv.take<int32_t>(R);
  t.rq_h = cv.take<int32_t>(R);
  t.rq_s = cv.take<int32_t>(R);
  t.rq_cbase = cv.take<int32_t>(R);
  t.rq_a = cv.take<int32_t>(R);
  t.rq_e = cv.take<int32_t>(R);
  t.rq_fu = cv.take<uint32_t>(R);
  t.rq_cid = cv.take<int32_t>(R);
  t.rq_hs = cv.take<uint32_t>(R);
  t.rq_p = cv.take<uint64_t>(R);
  t.rq_flags = cv.take<uint8_t>(R);
  t.rq_knew = cv.take<uint8_t>(R);
  t.pos_key = cv.take<uint64_t>(B);
  t.pos_req = cv.take<uint32_t>(B);
  t.pos_m = cv.take<uint32_t>(B);
  t.chunks = cv.take<ChunkDesc>((size_t)d.max_segments);
  t.val_tile = cv.take<uint64_t>(R / kValTile + 1);
  t.seg_word = cv.take<uint64_t>((size_t)d.max_segments);
  t.pos_blk = cv.take<uint32_t>(B);
  t.pos_claim = cv.take<uint32_t>(B);
  t.pos_elig = cv.take<uint8_t>(B);
  t.claims = cv.take<ClaimEntry>((size_t)kClaimWays << d.cl_log2);
  t.bm_victim = cv.take<uint32_t>((size_t)d.nwords);
  t.bm_inval = cv.take<uint32_t>((size_t)d.nwords);
  t.csk = cv.take<uint64_t>(N);
  t.grp_qsize = cv.take<int64_t>(G);
  t.grp_P = cv.take<int64_t>(G);
  t.grp_delta = cv.take<int64_t>(G);
  t.grp_x = cv.take<int64_t>(G);
  t.grp_pinned = cv.take<int64_t>(G);
  t.grp_full = cv.take<uint8_t>(G);
  t.sel = cv.take<SelSeg>(G);
  t.cls = cv.take<ClsRange>(G * kClasses);
  t.hist_bins = cv.take<uint32_t>(G * kRadixBins);
  {
    const size_t wrows = G < (size_t)kWideRows ? G : (size_t)kWideRows;
    const size_t wb = wrows * kWideBins > G * kRadixBins ? wrows * kWideBins : G * kRadixBins;
    t.wide_bins = cv.take<uint32_t>(wb);
  }
  t.wide_coarse = cv.take<uint32_t>((size_t)kWideRows * kRadixBins);
  t.wide_seg = cv.take<int16_t>(G);
  t.lst_key = cv.take<uint64_t>(N);
  t.lst_blk = cv.take<uint32_t>(N);
  t.lst_seg = cv.take<uint16_t>(N);
  t.bm_chunk_cnt = cv.take<int32_t>(3 * (((size_t)d.nwords + kBmChunk - 1) / kBmChunk));  // free, evicted, invalidated
  t.s3_attr = cv.take<uint8_t>(2 * (size_t)d.s3_np);
  t.s3_ck = cv.take<S3Chunk>(2 * (size_t)d.s3_nch);
  t.s3_base = cv.take<S3Base>(2 * (size_t)d.s3_nch);
  t.s3_rck = cv.take<uint32_t>((size_t)d.s3_nrch);
  t.s3_rbase = cv.take<uint32_t>((size_t)d.s3_nrch);
  t.s3_plan = cv.take<S3Plan>(1);
  t.s3_hit = cv.take<uint8_t>(B);
  t.s3_ick = cv.take<uint32_t>(B / kS3Chunk + 1);
  if (d.lg) {
    const size_t L = (size_t)d.lg_L;
    t.lg_L = d.lg_L;
    t.lg_P = d.lg_P;
    t.lg_max_chunks = d.lg_max_chunks;
    t.lg_app_chunks = d.lg_app_chunks;
    t.lg_blk = cv.take<uint32_t>(2 * (size_t)d.lg_P);
    t.lg_st = cv.take<uint64_t>(2 * (size_t)d.lg_P);
    t.lg_desc = cv.take<LogDesc>(L);
    t.lg_new = cv.take<LogDesc>(L);
    t.lg_live = cv.take<int64_t>(L);
    t.lg_add = cv.take<int64_t>(L);
    t.lg_pin = cv.take<int64_t>(L);
    t.lg_slot = cv.take<uint32_t>(B);
    t.lg_app = cv.take<uint32_t>(L * (size_t)d.lg_app_chunks);
    t.lg_tk = cv.take<LogTake>(L);
    t.lg_c0 = cv.take<int32_t>(L + 1);
    t.lg_ck = cv.take<uint32_t>((size_t)d.lg_max_chunks);
    t.lg_ck_out = cv.take<int64_t>((size_t)d.lg_max_chunks);
    t.lg_tie = cv.take<TieItem>(G);
  }
  StepArgs* step_args = cv.take<StepArgs>(1);
  // staging for ps_step_host
  ps_handle::Staging stg[2];
  for (auto& x : stg) {
    x.group = cv.take<int32_t>(R);
    x.offsets = cv.take<int64_t>(R + 1);
    x.tokens = cv.take<int32_t>((size_t)d.max_tokens);
    x.contract = cv.take<int32_t>(R);
    x.prefix = cv.take<uint64_t>(R);
  }
  ps_step_out_t so{};
  so.hit_blocks = cv.take<int32_t>(R);
  so.admitted_blocks = cv.take<int32_t>(R);
  so.admitted_offsets = cv.take<int32_t>(R + 1);
  so.admitted_ids = cv.take<int32_t>(B);
  so.evicted_ids = cv.take<int32_t>(B);
  so.invalidated_ids = cv.take<int32_t>(B);
  so.counts = cv.take<int32_t>(4);
  so.debt_raw = cv.take<int64_t>(G);
  so.debt_norm = cv.take<int64_t>(G);
  so.ids_capacity = (int64_t)B;
  so.req_capacity = (int32_t)R;
  const size_t total = align_up(cv.off, 256);
  if (base) {
    *s = t;
    h->stg[0] = stg[0];
    h->stg[1] = stg[1];
    h->st_out = so;
    h->step_args = step_args;
  }
  (void)zero_end;
  return total;
}

int32_t init_state(ps_handle* h, cudaStream_t st) {
  const DevState& s = h->base;
  // everything zero, then the non-zero patterns
  if (cudaMemsetAsync(h->workspace, 0, h->workspace_bytes, st) != cudaSuccess) return PS_ERR_CUDA;
  if (cudaMemsetAsync(s.table, 0xFF, sizeof(TableEntry) * ((size_t)kTableWays << s.tb_nbuckets_log2), st) != cudaSuccess)
    return PS_ERR_CUDA;
  if (cudaMemsetAsync(s.ghost_map, 0xFF, sizeof(TableEntry) * ((size_t)kTableWays << s.gh_nbuckets_log2), st) !=
      cudaSuccess)
    return PS_ERR_CUDA;
  launch_init(s, st);
  return cudaGetLastError() == cudaSuccess ? PS_OK : PS_ERR_CUDA;
}

inline cudaStream_t as_stream(void* p) { return reinterpret_cast<cudaStream_t>(p); }

// The stated sizes of a step's output arrays against what a step may write:
// B ids in each id list, R entries per request array.  Arrays left null (the
// host calls allow that) need no size.
bool capacities_ok(const ps_step_out_t& o, int64_t B, int32_t R) {
  const bool ids = o.admitted_ids || o.evicted_ids || o.invalidated_ids;
  const bool reqs = o.hit_blocks || o.admitted_blocks || o.admitted_offsets;
  return (!ids || o.ids_capacity >= B) && (!reqs || o.req_capacity >= R);
}

void drop_graph(ps_handle* h) {
  if (h->exec) cudaGraphExecDestroy(h->exec);
  if (h->graph) cudaGraphDestroy(h->graph);
  h->exec = nullptr;
  h->graph = nullptr;
}

// Capture the step's launch sequence once (its kernels read the per-step
// arguments from h->step_args, and every grid depends on the handle's bounds
// only); on any failure the handle keeps launching kernel by kernel.
void capture_step(ps_handle* h) {
  drop_graph(h);
  DevState tmpl = h->base;
  tmpl.args = h->step_args;
  tmpl.R = 0;
  bool ok = cudaStreamBeginCapture(h->cap_stream, cudaStreamCaptureModeThreadLocal) == cudaSuccess;
  if (ok) {
    const CaptureCtx ctx{h->cap_aux, h->cap_aux2, h->cap_side, h->cap_fork, h->cap_join,
                         h->cap_side2, h->cap_fork2, h->cap_join2};
    const int32_t rc = launch_step(tmpl, h->cap_stream, &h->trace, &ctx);
    // a body whose capture did not close leaves an auxiliary stream capturing
    // (the side stream joined the main capture: it ends with it)
    for (cudaStream_t a : {h->cap_aux2, h->cap_aux}) {
      cudaStreamCaptureStatus aux_cs = cudaStreamCaptureStatusNone;
      if (cudaStreamIsCapturing(a, &aux_cs) == cudaSuccess && aux_cs != cudaStreamCaptureStatusNone) {
        cudaGraph_t body = nullptr;
        cudaStreamEndCapture(a, &body);
      }
    }
    cudaGraph_t g = nullptr;
    const bool ended = cudaStreamEndCapture(h->cap_stream, &g) == cudaSuccess;
    ok = rc == PS_OK && ended && g;
    if (ok) {
      h->graph = g;
      ok = cudaGraphInstantiate(&h->exec, g, 0) == cudaSuccess;
    } else if (g) {
      cudaGraphDestroy(g);
    }
  }
  cudaGetLastError();  // a failed capture leaves no sticky launch error behind
  if (!ok) {
    drop_graph(h);
    h->use_graph = false;
  }
  h->exec_timing = h->trace.timing;
}

}  // namespace

namespace ps {
// Device state of a handle, for entry points defined outside this file.
const DevState* handle_state(const ps_handle_t* h) { return &h->base; }
}  // namespace ps

extern "C" {

size_t ps_workspace_bytes(int64_t capacity_blocks, int32_t block_size, int32_t num_groups, const ps_params_t* params,
                          int32_t max_requests, int64_t max_tokens) {
  if (check_params(capacity_blocks, block_size, num_groups, 0, params) != PS_OK) return 0;
  if (max_requests < 0 || max_requests > PS_MAX_REQUESTS_PER_STEP || max_tokens < 0 || max_tokens > (1ll << 31))
    return 0;
  const Dims d = make_dims(capacity_blocks, block_size, num_groups, params, max_requests, max_tokens);
  return carve(d, nullptr, nullptr, nullptr);
}

int32_t ps_create(ps_handle_t** out, int64_t capacity_blocks, int32_t block_size, int32_t num_groups, int32_t policy,
                  const ps_params_t* params, void* d_workspace, size_t workspace_bytes, int32_t max_requests,
                  int64_t max_tokens, void* stream) {
  if (!out) return PS_ERR_INVALID_ARG;
  *out = nullptr;
  if (check_params(capacity_blocks, block_size, num_groups, policy, params) != PS_OK) return PS_ERR_INVALID_ARG;
  const size_t need = ps_workspace_bytes(capacity_blocks, block_size, num_groups, params, max_requests, max_tokens);
  if (need == 0 || !d_workspace || workspace_bytes < need || (reinterpret_cast<uintptr_t>(d_workspace) & 255))
    return PS_ERR_INVALID_ARG;
  ps_handle* h = new (std::nothrow) ps_handle();
  if (!h) return PS_ERR_INVALID_ARG;
  const Dims d = make_dims(capacity_blocks, block_size, num_groups, params, max_requests, max_tokens);
  h->workspace = d_workspace;
  h->workspace_bytes = need;
  cudaGetDevice(&h->device);
  DevState s{};
  carve(d, static_cast<char*>(d_workspace), &s, h);
  s.N = capacity_blocks; s.bs = block_size; s.G = num_groups; s.C = params->num_contracts; s.policy = policy;
  s.flags = params->flags; s.fp_shift = params->fp_shift; s.eps = params->epsilon_fp; s.hash_seed = params->hash_seed;
  s.lg_on = d.lg && policy != PS_S3FIFO;
  s.rho_min = params->rho_fp[0];
  for (int c = 0; c < PS_MAX_CONTRACTS; ++c) {
    s.rho[c] = c < s.C ? params->rho_fp[c] : 1;
    s.beta[c] = c < s.C ? params->beta_fp[c] : 0;
    if (c < s.C && params->rho_fp[c] < s.rho_min) s.rho_min = params->rho_fp[c];
  }
  s.s3_small_pct = params->s3_small_pct; s.s3_freq_cap = params->s3_freq_cap; s.s3_move_min = params->s3_move_min_freq;
  s.s3_small_cap = d.s3_small_cap; s.s3_ghost_cap = d.s3_ghost_cap;
  s.gh_nbuckets_log2 = d.gh_log2; s.ghost_ring_cap = d.ghost_ring_cap;
  s.s3_np = d.s3_np; s.s3_nch = d.s3_nch; s.s3_nrch = d.s3_nrch;
  s.max_requests = max_requests; s.max_tokens = max_tokens; s.max_blocks = d.max_blocks;
  s.history_capacity = params->history_capacity;
  s.tb_nbuckets_log2 = d.tb_log2; s.cl_nbuckets_log2 = d.cl_log2; s.hist_cap_log2 = d.hist_log2;
  s.nwords = d.nwords;
  s.max_segments = d.max_segments;
  const KeySchedule ks = key_schedule(params->hash_seed, block_size);
  s.chain_mul = ks.kc;
  s.digest_mul = ks.kd;
  s.args = h->step_args;
  h->base = s;
  h->contract_of_group.assign(params->contract_of_group, params->contract_of_group + num_groups);
  cudaStream_t st = as_stream(stream);
  configure_kernels(s);  // per device: attributes are set on the current one
  int32_t rc = init_state(h, st);
  if (rc == PS_OK) rc = upload_constants(h, st);
  if (rc == PS_OK && (cudaStreamCreateWithFlags(&h->cap_stream, cudaStreamNonBlocking) != cudaSuccess ||
                      cudaStreamCreateWithFlags(&h->cap_aux, cudaStreamNonBlocking) != cudaSuccess ||
                      cudaStreamCreateWithFlags(&h->cap_aux2, cudaStreamNonBlocking) != cudaSuccess ||
                      cudaStreamCreateWithFlags(&h->cap_side, cudaStreamNonBlocking) != cudaSuccess ||
                      cudaStreamCreateWithFlags(&h->cap_side2, cudaStreamNonBlocking) != cudaSuccess ||
                      cudaEventCreateWithFlags(&h->cap_fork, cudaEventDisableTiming) != cudaSuccess ||
                      cudaEventCreateWithFlags(&h->cap_join, cudaEventDisableTiming) != cudaSuccess ||
                      cudaEventCreateWithFlags(&h->cap_fork2, cudaEventDisableTiming) != cudaSuccess ||
                      cudaEventCreateWithFlags(&h->cap_join2, cudaEventDisableTiming) != cudaSuccess ||
                      cudaStreamCreateWithFlags(&h->copy_stream, cudaStreamNonBlocking) != cudaSuccess))
    rc = PS_ERR_CUDA;
  for (int k = 0; k < 2 && rc == PS_OK; ++k)
    if (cudaEventCreateWithFlags(&h->in_ready[k], cudaEventDisableTiming) != cudaSuccess ||
        cudaEventCreateWithFlags(&h->slot_free[k], cudaEventDisableTiming) != cudaSuccess ||
        cudaEventCreateWithFlags(&h->done[k], cudaEventDisableTiming) != cudaSuccess)
    rc = PS_ERR_CUDA;
  if (rc != PS_OK) {
    delete h;
    return rc;
  }
  *out = h;
  return PS_OK;
}

int32_t ps_step(ps_handle_t* h, void* stream, int64_t now_ticks, int32_t num_requests, const int32_t* d_group_ids,
                const int64_t* d_token_offsets, const int32_t* d_tokens, const int32_t* d_contract_ids,
                const uint64_t* d_prefix_ids, const ps_step_out_t* out) {
  if (!h || !out || num_requests < 0 || num_requests > h->base.max_requests || !d_token_offsets) return PS_ERR_INVALID_ARG;
  if (num_requests > 0 && (!d_group_ids || !d_tokens)) return PS_ERR_INVALID_ARG;
  if (!out->hit_blocks || !out->admitted_blocks || !out->admitted_offsets || !out->admitted_ids || !out->evicted_ids ||
      !out->invalidated_ids || !out->counts || !out->debt_raw || !out->debt_norm ||
      !capacities_ok(*out, h->base.max_blocks, num_requests))
    return PS_ERR_INVALID_ARG;
  DevState s = h->base;
  s.now = now_ticks;
  s.R = num_requests;
  s.in_group = d_group_ids;
  s.in_offsets = d_token_offsets;
  s.in_tokens = d_tokens;
  s.in_contract = d_contract_ids;
  s.in_prefix = d_prefix_ids;
  s.tokens_aligned16 = (reinterpret_cast<uintptr_t>(d_tokens) & 15) == 0;
  s.out = *out;
  s.args = h->step_args;
  cudaStream_t st = as_stream(stream);
  const StepArgs a = args_of(s);
  if (cudaMemcpyAsync(h->step_args, &a, sizeof(a), cudaMemcpyHostToDevice, st) != cudaSuccess) return PS_ERR_CUDA;
  if (h->use_graph && (!h->exec || h->exec_timing != h->trace.timing)) capture_step(h);
  if (h->use_graph && h->exec)
    return cudaGraphLaunch(h->exec, st) == cudaSuccess ? PS_OK : PS_ERR_CUDA;
  return launch_step(s, st, &h->trace);
}

int32_t ps_step_host(ps_handle_t* h, void* stream, int64_t now_ticks, int32_t num_requests, const int32_t* h_group_ids,
                     const int64_t* h_token_offsets, const int32_t* h_tokens, const int32_t* h_contract_ids,
                     const uint64_t* h_prefix_ids, const ps_host_out_t* h_out) {
  if (!h || !h_out || num_requests < 0 || num_requests > h->base.max_requests || !h_token_offsets)
    return PS_ERR_INVALID_ARG;
  const int64_t T = num_requests > 0 ? h_token_offsets[num_requests] : 0;
  if (T < 0 || T > h->base.max_tokens || (num_requests > 0 && (!h_group_ids || (T > 0 && !h_tokens))) ||
      !capacities_ok(*h_out, h->base.max_blocks, num_requests))
    return PS_ERR_INVALID_ARG;
  cudaStream_t st = as_stream(stream);
  const size_t R = (size_t)num_requests;
  auto h2d = [&](void* d, const void* src, size_t bytes) {
    return bytes == 0 || cudaMemcpyAsync(d, src, bytes, cudaMemcpyHostToDevice, st) == cudaSuccess;
  };
  const ps_handle::Staging& sg = h->stg[0];
  if (!h2d(sg.offsets, h_token_offsets, (R + 1) * 8) || !h2d(sg.group, h_group_ids, R * 4) ||
      !h2d(sg.tokens, h_tokens, (size_t)T * 4) || (h_contract_ids && !h2d(sg.contract, h_contract_ids, R * 4)) ||
      (h_prefix_ids && !h2d(sg.prefix, h_prefix_ids, R * 8)))
    return PS_ERR_CUDA;
  int32_t rc = ps_step(h, stream, now_ticks, num_requests, sg.group, sg.offsets, sg.tokens,
                       h_contract_ids ? sg.contract : nullptr, h_prefix_ids ? sg.prefix : nullptr, &h->st_out);
  if (rc != PS_OK) return rc;
  const ps_step_out_t& o = h->st_out;
  auto d2h = [&](void* dst, const void* d, size_t bytes) {
    return bytes == 0 || !dst || cudaMemcpyAsync(dst, d, bytes, cudaMemcpyDeviceToHost, st) == cudaSuccess;
  };
  const size_t G = (size_t)h->base.G;
  if (!d2h(h_out->counts, o.counts, 16) || !d2h(h_out->hit_blocks, o.hit_blocks, R * 4) ||
      !d2h(h_out->admitted_blocks, o.admitted_blocks, R * 4) ||
      !d2h(h_out->admitted_offsets, o.admitted_offsets, (R + 1) * 4) || !d2h(h_out->debt_raw, o.debt_raw, G * 8) ||
      !d2h(h_out->debt_norm, o.debt_norm, G * 8) || cudaStreamSynchronize(st) != cudaSuccess)
    return PS_ERR_CUDA;
  if (!h_out->counts || h_out->counts[3] != PS_OK) return h_out->counts ? h_out->counts[3] : PS_OK;
  if (!d2h(h_out->admitted_ids, o.admitted_ids, (size_t)h_out->counts[0] * 4) ||
      !d2h(h_out->evicted_ids, o.evicted_ids, (size_t)h_out->counts[1] * 4) ||
      !d2h(h_out->invalidated_ids, o.invalidated_ids, (size_t)h_out->counts[2] * 4) ||
      cudaStreamSynchronize(st) != cudaSuccess)
    return PS_ERR_CUDA;
  return PS_OK;
}

namespace {
// A host array a kernel may write: page-locked (or otherwise device-mapped).
bool device_writable(const void* p) {
  if (!p) return true;
  cudaPointerAttributes a{};
  if (cudaPointerGetAttributes(&a, p) != cudaSuccess) {
    cudaGetLastError();
    return false;
  }
  return a.type == cudaMemoryTypeHost || a.type == cudaMemoryTypeManaged;
}
}  // namespace

int32_t ps_step_host_async(ps_handle_t* h, void* stream, int32_t slot, int64_t now_ticks, int32_t num_requests,
                           const int32_t* h_group_ids, const int64_t* h_token_offsets, const int32_t* h_tokens,
                           const int32_t* h_contract_ids, const uint64_t* h_prefix_ids, const ps_host_out_t* h_out) {
  if (!h || !h_out || slot < 0 || slot > 1 || h->pending[slot] || num_requests < 0 ||
      num_requests > h->base.max_requests || !h_token_offsets || !h_out->counts)
    return PS_ERR_INVALID_ARG;
  const int64_t T = num_requests > 0 ? h_token_offsets[num_requests] : 0;
  if (T < 0 || T > h->base.max_tokens || (num_requests > 0 && (!h_group_ids || (T > 0 && !h_tokens))) ||
      !capacities_ok(*h_out, h->base.max_blocks, num_requests))
    return PS_ERR_INVALID_ARG;
  for (const void* p : {(const void*)h_out->hit_blocks, (const void*)h_out->admitted_blocks,
                        (const void*)h_out->admitted_offsets, (const void*)h_out->admitted_ids,
                        (const void*)h_out->evicted_ids, (const void*)h_out->invalidated_ids,
                        (const void*)h_out->counts, (const void*)h_out->debt_raw, (const void*)h_out->debt_norm})
    if (!device_writable(p)) return PS_ERR_INVALID_ARG;
  cudaStream_t st = as_stream(stream), cs = h->copy_stream;
  const size_t R = (size_t)num_requests;
  const ps_handle::Staging& sg = h->stg[slot];
  auto h2d = [&](void* d, const void* src, size_t bytes) {
    return bytes == 0 || cudaMemcpyAsync(d, src, bytes, cudaMemcpyHostToDevice, cs) == cudaSuccess;
  };
  // the slot's staging is free once the step that last read it has run
  if (cudaStreamWaitEvent(cs, h->slot_free[slot], 0) != cudaSuccess) return PS_ERR_CUDA;
  if (!h2d(sg.offsets, h_token_offsets, (R + 1) * 8) || !h2d(sg.group, h_group_ids, R * 4) ||
      !h2d(sg.tokens, h_tokens, (size_t)T * 4) || (h_contract_ids && !h2d(sg.contract, h_contract_ids, R * 4)) ||
      (h_prefix_ids && !h2d(sg.prefix, h_prefix_ids, R * 8)) ||
      cudaEventRecord(h->in_ready[slot], cs) != cudaSuccess || cudaStreamWaitEvent(st, h->in_ready[slot], 0) != cudaSuccess)
    return PS_ERR_CUDA;
  const int32_t rc = ps_step(h, stream, now_ticks, num_requests, sg.group, sg.offsets, sg.tokens,
                             h_contract_ids ? sg.contract : nullptr, h_prefix_ids ? sg.prefix : nullptr, &h->st_out);
  if (rc != PS_OK) return rc;
  if (cudaEventRecord(h->slot_free[slot], st) != cudaSuccess) return PS_ERR_CUDA;
  launch_host_out(h->st_out, *h_out, num_requests, h->base.G, st);
  if (cudaGetLastError() != cudaSuccess || cudaEventRecord(h->done[slot], st) != cudaSuccess) return PS_ERR_CUDA;
  h->pending[slot] = h_out;
  return PS_OK;
}

int32_t ps_step_host_wait(ps_handle_t* h, int32_t slot) {
  if (!h || slot < 0 || slot > 1 || !h->pending[slot]) return PS_ERR_INVALID_ARG;
  const ps_host_out_t* o = h->pending[slot];
  h->pending[slot] = nullptr;
  if (cudaEventSynchronize(h->done[slot]) != cudaSuccess) return PS_ERR_CUDA;
  return o->counts[3];
}

int32_t ps_stats(ps_handle_t* h, void* stream, int64_t* h_stats) {
  if (!h || !h_stats) return PS_ERR_INVALID_ARG;
  cudaStream_t st = as_stream(stream);
  int32_t sticky = PS_OK;
  if (cudaMemcpyAsync(h_stats, h->base.stats, sizeof(int64_t) * h->base.G * PS_NUM_STATS, cudaMemcpyDeviceToHost, st) !=
          cudaSuccess ||
      cudaMemcpyAsync(&sticky, &h->base.ctl->sticky, 4, cudaMemcpyDeviceToHost, st) != cudaSuccess ||
      cudaStreamSynchronize(st) != cudaSuccess)
    return PS_ERR_CUDA;
  return sticky;
}

int32_t ps_clear_status(ps_handle_t* h, void* stream) {
  if (!h) return PS_ERR_INVALID_ARG;
  return cudaMemsetAsync(&h->base.ctl->sticky, 0, 4, as_stream(stream)) == cudaSuccess ? PS_OK : PS_ERR_CUDA;
}

int32_t ps_reset(ps_handle_t* h, void* stream) {
  if (!h) return PS_ERR_INVALID_ARG;
  cudaStream_t st = as_stream(stream);
  const int32_t rc = init_state(h, st);
  return rc != PS_OK ? rc : upload_constants(h, st);
}

int32_t ps_cached_prefix(ps_handle_t* h, void* stream, int32_t num_requests, const int32_t* d_group_ids,
                         const int64_t* d_token_offsets, const int32_t* d_tokens, int32_t* d_cached_blocks,
                         int32_t* d_status) {
  if (!h || num_requests < 0 || num_requests > h->base.max_requests || !d_token_offsets || !d_status)
    return PS_ERR_INVALID_ARG;
  if (num_requests > 0 && (!d_group_ids || !d_tokens || !d_cached_blocks)) return PS_ERR_INVALID_ARG;
  DevState s = h->base;
  s.R = num_requests;
  s.in_group = d_group_ids;
  s.in_offsets = d_token_offsets;
  s.in_tokens = d_tokens;
  s.in_contract = nullptr;
  s.in_prefix = nullptr;
  s.tokens_aligned16 = (reinterpret_cast<uintptr_t>(d_tokens) & 15) == 0;
  return launch_probe(s, as_stream(stream), d_cached_blocks, d_status);
}

void ps_destroy(ps_handle_t* h) {
  if (!h) return;
  drop_graph(h);
  if (h->cap_stream) cudaStreamDestroy(h->cap_stream);
  if (h->cap_aux) cudaStreamDestroy(h->cap_aux);
  if (h->cap_aux2) cudaStreamDestroy(h->cap_aux2);
  if (h->cap_side) cudaStreamDestroy(h->cap_side);
  if (h->cap_side2) cudaStreamDestroy(h->cap_side2);
  if (h->cap_fork) cudaEventDestroy(h->cap_fork);
  if (h->cap_join) cudaEventDestroy(h->cap_join);
  if (h->cap_fork2) cudaEventDestroy(h->cap_fork2);
  if (h->cap_join2) cudaEventDestroy(h->cap_join2);
  if (h->copy_stream) cudaStreamDestroy(h->copy_stream);
  for (int k = 0; k < 2; ++k)
    for (cudaEvent_t e : {h->in_ready[k], h->slot_free[k], h->done[k]})
      if (e) cudaEventDestroy(e);
  if (h->trace.timing)
    for (cudaEvent_t e : h->trace.ev) cudaEventDestroy(e);
  delete h;
}

int32_t ps_set_stage_timing(ps_handle_t* h, int32_t enable) {
  if (!h) return PS_ERR_INVALID_ARG;
  if (enable && !h->trace.timing) {
    for (cudaEvent_t& e : h->trace.ev)
      if (cudaEventCreate(&e) != cudaSuccess) return PS_ERR_CUDA;
    h->trace.timing = true;
  } else if (!enable && h->trace.timing) {
    drop_graph(h);  // its event nodes refer to the events
    for (cudaEvent_t e : h->trace.ev) cudaEventDestroy(e);
    h->trace.timing = false;
  }
  return PS_OK;
}

int32_t ps_get_stage_times(ps_handle_t* h, float* h_ms, int32_t max_stages, int32_t* h_launches) {
  if (!h || (!h_ms && max_stages > 0)) return PS_ERR_INVALID_ARG;
  if (h_launches) *h_launches = h->trace.launches;
  if (!h->trace.timing) return 0;
  if (cudaEventSynchronize(h->trace.ev[PS_NUM_STAGES]) != cudaSuccess) return PS_ERR_CUDA;
  // kernels the step actually launched (conditional bodies included or not)
  if (h_launches && cudaMemcpy(h_launches, &h->base.ctl->nlaunch, 4, cudaMemcpyDeviceToHost) != cudaSuccess)
    return PS_ERR_CUDA;
  const int n = max_stages < PS_NUM_STAGES ? max_stages : PS_NUM_STAGES;
  for (int k = 0; k < n; ++k)
    if (cudaEventElapsedTime(h_ms + k, h->trace.ev[k], h->trace.ev[k + 1]) != cudaSuccess) return PS_ERR_CUDA;
  return n;
}

int32_t ps_set_graph(ps_handle_t* h, int32_t enable) {
  if (!h) return PS_ERR_INVALID_ARG;
  if (!enable) drop_graph(h);
  h->use_graph = enable != 0;  // captured (again) at the next step
  return PS_OK;
}

int32_t ps_uses_graph(const ps_handle_t* h) {
  if (!h) return PS_ERR_INVALID_ARG;
  return h->use_graph && h->exec ? 1 : 0;
}

const char* ps_status_string(int32_t status) {
  switch (status) {
    case PS_OK: return "ok";
    case PS_ERR_INVALID_ARG: return "invalid argument";
    case PS_ERR_CAPACITY: return "capacity exceeded";
    case PS_ERR_CLOCK: return "accounting clock went backwards";
    case PS_ERR_CUDA: return "CUDA error";
    case PS_ERR_TIMEOUT: return "device wait timed out";
    case PS_ERR_DEVICE_STATUS: return "device reported an error";
    default: return "unknown status";
  }
}

int32_t ps_export_state(ps_handle_t* h, void* stream, ps_state_view_t* v) {
  if (!h || !v) return PS_ERR_INVALID_ARG;
  cudaStream_t st = as_stream(stream);
  const DevState& s = h->base;
  const size_t N = (size_t)s.N;
  std::vector<uint8_t> flags(N), contract(N), klass(N);
  std::vector<uint16_t> group(N);
  std::vector<uint32_t> freq(N);
  Ctl ctl{};
  bool ok = true;
  auto d2h = [&](void* dst, const void* src, size_t bytes) {
    ok = ok && cudaMemcpyAsync(dst, src, bytes, cudaMemcpyDeviceToHost, st) == cudaSuccess;
  };
  d2h(flags.data(), s.blk_flags, N);
  d2h(contract.data(), s.blk_contract, N);
  d2h(klass.data(), s.blk_klass, N);
  d2h(group.data(), s.blk_group, N * 2);
  d2h(freq.data(), s.blk_freq, N * 4);
  d2h(&ctl, s.ctl, sizeof(Ctl));
  if (v->key) d2h(v->key, s.blk_key, N * 8);
  if (v->prefix) d2h(v->prefix, s.blk_prefix, N * 8);
  if (v->stamp) d2h(v->stamp, s.blk_stamp, N * 8);
  if (v->acc) d2h(v->acc, s.blk_acc, N * 4);
  if (v->s3seq) d2h(v->s3seq, s.blk_s3seq, N * 8);
  if (v->balances) d2h(v->balances, s.ledger, sizeof(int64_t) * s.G * s.C);
  if (!ok || cudaStreamSynchronize(st) != cudaSuccess) return PS_ERR_CUDA;
  for (size_t b = 0; b < N; ++b) {
    if (v->resident) v->resident[b] = flags[b] & 1;
    if (v->group) v->group[b] = group[b];
    if (v->contract) v->contract[b] = contract[b];
    if (v->klass) v->klass[b] = klass[b];
    if (v->freq) v->freq[b] = (int32_t)(freq[b] < (uint32_t)s.s3_freq_cap ? freq[b] : (uint32_t)s.s3_freq_cap);
    if (v->s3q) v->s3q[b] = (flags[b] >> 1) & 1;
  }
  v->t_prev = ctl.t_prev;
  v->step = ctl.step;
  v->s3_ctr = ctl.s3_ctr;
  v->ghost_ctr = ctl.ghost_ctr;
  return PS_OK;
}

int64_t ps_export_history(ps_handle_t* h, void* stream, int32_t* h_group, uint64_t* h_prefix, uint64_t* h_refcount,
                          uint8_t* h_admitted, int64_t cap) {
  if (!h) return PS_ERR_INVALID_ARG;
  cudaStream_t st = as_stream(stream);
  const size_t n = (size_t)1 << h->base.hist_cap_log2;
  std::vector<HistEntry> e(n);
  if (cudaMemcpyAsync(e.data(), h->base.hist, n * sizeof(HistEntry), cudaMemcpyDeviceToHost, st) != cudaSuccess ||
      cudaStreamSynchronize(st) != cudaSuccess)
    return PS_ERR_CUDA;
  int64_t k = 0;
  for (const HistEntry& x : e) {
    if (x.g1 == 0) continue;  // every installed entry, so a failed step's leftovers would show
    const uint32_t rc = x.refadm & 0x7FFFFFFFu;
    const bool adm = x.refadm >> 31;
    if (h_group && k < cap) {
      h_group[k] = (int32_t)x.g1 - 1;
      h_prefix[k] = x.p;
      h_refcount[k] = rc;
      h_admitted[k] = adm;
    }
    ++k;
  }
  return k;
}

int64_t ps_export_ghost(ps_handle_t* h, void* stream, int32_t* h_group, uint64_t* h_key, uint64_t* h_seq, int64_t cap) {
  if (!h) return PS_ERR_INVALID_ARG;
  cudaStream_t st = as_stream(stream);
  const DevState& s = h->base;
  // copy the ghost map and each slot's sequence number, read them here
  const size_t n = (size_t)kTableWays << s.gh_nbuckets_log2;
  std::vector<TableEntry> map(n);
  std::vector<uint64_t> seq(n);
  if (cudaMemcpyAsync(map.data(), s.ghost_map, n * sizeof(TableEntry), cudaMemcpyDeviceToHost, st) != cudaSuccess ||
      cudaMemcpyAsync(seq.data(), s.ghost_sq, n * 8, cudaMemcpyDeviceToHost, st) != cudaSuccess ||
      cudaStreamSynchronize(st) != cudaSuccess)
    return PS_ERR_CUDA;
  int64_t k = 0;
  for (size_t i = 0; i < n; ++i) {
    const TableEntry& e = map[i];
    if (e.blk == kNone) continue;
    if (h_group && k < cap) {
      h_group[k] = (int32_t)e.grp;
      h_key[k] = e.key;
      h_seq[k] = seq[i];
    }
    ++k;
  }
  return k;
}

}  // extern "C"
