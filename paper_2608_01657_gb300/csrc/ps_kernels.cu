// Kernels of the batched prefix-cache step (PrefixShield, arXiv 2608.01657).
//
// One step is a fixed sequence of launches on the caller's stream.  Nothing on
// the path goes back to the host: every size (tokens, blocks, claims, victims)
// lives in device memory, grids are sized from the handle's bounds, and a
// thread whose item does not exist exits at once.  Apart from the one-CTA
// scans, every stage runs a thread per block position, per request or per
// victim, so a long prompt is spread over many warps instead of serializing
// one.  Each kernel's comment names the stage and the passage it implements.
#include <climits>
#include <cstdio>

#include <vector>

#include "ps_device.cuh"
#include "ps_launch.cuh"

namespace ps {

constexpr int kFinCap = 8192;  // split lists up to this size are finished by one CTA in shared memory
constexpr int kFinRows = 32;   // rows k_list_finish counts at once (32 KB)
constexpr int kFinCountCap = 512;  // split lists up to this size are ranked by counting

// 128-bit compare-and-swap (sm_90+): installs the (p, group) identity of a
// history entry atomically, so two requests of one (group, prefix) that race
// to insert it agree on the slot.
__device__ __forceinline__ void cas128(void* addr, uint64_t exp_lo, uint64_t exp_hi, uint64_t new_lo,
                                       uint64_t new_hi, uint64_t* old_lo, uint64_t* old_hi) {
  uint64_t lo, hi;
  asm volatile(
      "{\n\t.reg .b128 e, n, d;\n\t"
      "mov.b128 e, {%2, %3};\n\t"
      "mov.b128 n, {%4, %5};\n\t"
      "atom.global.cas.b128 d, [%6], e, n;\n\t"
      "mov.b128 {%0, %1}, d;\n\t}"
      : "=l"(lo), "=l"(hi)
      : "l"(exp_lo), "l"(exp_hi), "l"(new_lo), "l"(new_hi), "l"(addr)
      : "memory");
  *old_lo = lo;
  *old_hi = hi;
}

__device__ __forceinline__ uint64_t step_tag(uint64_t step, uint32_t req) {
  return (step << 32) | (uint64_t)(0xFFFFFFFFu - req);
}
// The request index stored in a step tag, or UINT32_MAX if the tag is older.
__device__ __forceinline__ uint32_t tag_req(uint64_t tag, uint64_t step) {
  return (tag >> 32) == step ? 0xFFFFFFFFu - (uint32_t)tag : 0xFFFFFFFFu;
}
__device__ __forceinline__ int64_t refill(int64_t b, int64_t beta, int64_t rho, int64_t dt) {
  // Eq. 1, min{beta, b + rho*dt}, without overflow (dt >= ceil(need/rho) saturates).
  const int64_t need = beta - b;
  if (need <= 0 || dt >= (need + rho - 1) / rho) return beta;
  return b + rho * dt;
}
__device__ __forceinline__ int64_t muldiv(int64_t a, int64_t b, int64_t c) {
  return (int64_t)(((__int128)a * (__int128)b) / (__int128)c);
}

// ---- arithmetic modulo p = 2^61 - 1 (Mersenne reduction: 2^61 == 1) ------
__device__ __forceinline__ uint64_t red61(uint64_t x) {  // any 64-bit x -> [0, p)
  const uint64_t r = (x & kP61) + (x >> 61);
  return r >= kP61 ? r - kP61 : r;
}
__device__ __forceinline__ uint64_t add61(uint64_t a, uint64_t b) {  // a, b < p
  const uint64_t r = a + b;
  return r >= kP61 ? r - kP61 : r;
}
__device__ __forceinline__ uint64_t mul61(uint64_t a, uint64_t b) {  // a, b < p
  const uint64_t lo = a * b, hi = __umul64hi(a, b);
  uint64_t r = (lo & kP61) + ((lo >> 61) | (hi << 3));
  r = (r & kP61) + (r >> 61);
  return r >= kP61 ? r - kP61 : r;
}

// ---- native prefix table ---------------------------------------------------
// Lookup by one thread: the 128-byte home bucket (8 entries), then following
// buckets while the overflow count says some key probed past.
// All eight ways and the overflow count are loaded before any is compared,
// so a bucket costs one round trip (a return inside the loads would keep the
// compiler from issuing a later way's load before an earlier way's compare).
__device__ uint32_t table_find(const DevState& s, uint64_t key, uint32_t g) {
  const uint32_t mask = (1u << s.tb_nbuckets_log2) - 1;
  uint32_t b = table_home(key, g, s.tb_nbuckets_log2);
  for (uint32_t it = 0; it <= mask; ++it) {
    const uint4* e = reinterpret_cast<const uint4*>(s.table + (size_t)b * kTableWays);
    uint4 raw[kTableWays];
#pragma unroll
    for (int w = 0; w < kTableWays; ++w) raw[w] = __ldg(e + w);
    const uint32_t ovf = __ldg(s.table_ovf + b);  // issued with the bucket: a miss needs no second trip
    uint32_t hit = kNone;
#pragma unroll
    for (int w = 0; w < kTableWays; ++w)
      if (raw[w].z != kNone && raw[w].x == (uint32_t)key && raw[w].y == (uint32_t)(key >> 32) && raw[w].w == g)
        hit = raw[w].z;
    if (hit != kNone || ovf == 0) return hit;
    b = (b + 1) & mask;
  }
  return kNone;
}

// Returns the slot, with kDisplaced set when it lies past the home bucket
// (then a delete must repair the overflow counters on the way).  The swap
// starts at a way chosen by the key's own bits: at a quarter load that way
// is usually free, so most inserts take one atomic and no load.  (No key is
// inserted twice, so no swaps pile up on one way.)
constexpr uint32_t kDisplaced = 0x80000000u;
__device__ uint32_t table_insert(const DevState& s, uint64_t key, uint32_t g, uint32_t blk) {
  const uint32_t mask = (1u << s.tb_nbuckets_log2) - 1;
  uint32_t b = table_home(key, g, s.tb_nbuckets_log2);
  const uint32_t w0 = (uint32_t)(key >> 7) & (kTableWays - 1);
  for (uint32_t it = 0; it <= mask; ++it) {
    TableEntry* e = s.table + (size_t)b * kTableWays;
    for (int q = 0; q < kTableWays; ++q) {
      const int w = (int)((w0 + (uint32_t)q) & (kTableWays - 1));
      if (atomicCAS(&e[w].blk, kNone, blk) == kNone) {
        e[w].key = key;
        e[w].grp = g;
        return (b * kTableWays + w) | (it ? kDisplaced : 0u);
      }
    }
    atomicAdd(s.table_ovf + b, 1u);
    b = (b + 1) & mask;
  }
  return kNone;  // unreachable: the table is at most a quarter full
}

// An entry is empty exactly when its block field is kNone (lookups test it
// first), so a delete clears only that field: an insert that takes the slot
// at once then writes its own key and group, and no late clearing store of
// the delete can land on them.
// The same from the block's record as already loaded (slot with its flag,
// key, group).
__device__ __forceinline__ void table_delete_known(const DevState& s, uint32_t tagged, uint64_t key, uint32_t g) {
  const uint32_t mask = (1u << s.tb_nbuckets_log2) - 1;
  const uint32_t slot = tagged & ~kDisplaced;
  s.table[slot].blk = kNone;
  if (!(tagged & kDisplaced)) return;  // in its home bucket: no counter passed
  const uint32_t bucket = slot / kTableWays;
  uint32_t x = table_home(key, g, s.tb_nbuckets_log2);
  for (uint32_t it = 0; x != bucket && it <= mask; ++it, x = (x + 1) & mask) atomicSub(s.table_ovf + x, 1u);
}
__device__ void table_delete(const DevState& s, uint32_t blk) {
  const uint32_t mask = (1u << s.tb_nbuckets_log2) - 1;
  const uint32_t tagged = s.blk_slot[blk];
  const uint32_t slot = tagged & ~kDisplaced;
  s.table[slot].blk = kNone;
  if (!(tagged & kDisplaced)) return;  // in its home bucket: no counter passed
  const uint32_t bucket = slot / kTableWays;
  uint32_t x = table_home(s.blk_key[blk], s.blk_group[blk], s.tb_nbuckets_log2);
  for (uint32_t it = 0; x != bucket && it <= mask; ++it, x = (x + 1) & mask) atomicSub(s.table_ovf + x, 1u);
}

// ---- per-step claim map ------------------------------------------------------
// The bucket's keys are loaded first, so the many requests that claim one
// popular key in a step mostly find it with a plain load and swap nothing
// (a swap first would serialize them on one address).
__device__ uint32_t claim_insert(const DevState& s, uint64_t key, uint32_t req) {
  const uint32_t mask = (1u << s.cl_nbuckets_log2) - 1;
  uint32_t b = claim_home(key, s.cl_nbuckets_log2);
  for (uint32_t it = 0; it <= mask; ++it) {
    // the bucket's keys in one round of loads.  Keys only arrive during a
    // step, each in the first free way, so walking the ways in order with a
    // CAS on each free one meets the key wherever another thread put it.
    ClaimEntry* e = s.claims + (size_t)b * kClaimWays;
    uint64_t cur[kClaimWays];
#pragma unroll
    for (int w = 0; w < kClaimWays; ++w) cur[w] = ldcg_u64(&e[w].key);
#pragma unroll
    for (int w = 0; w < kClaimWays; ++w) {
      uint64_t v = cur[w];
      if (v == 0) v = atomicCAS(reinterpret_cast<unsigned long long*>(&e[w].key), 0ull, (unsigned long long)key);
      if (v == 0 || v == key) {
        atomicMin(&e[w].minreq, req);
        return b * kClaimWays + w;
      }
    }
    b = (b + 1) & mask;
  }
  return kNone;  // unreachable: the map has a slot for every block of a step
}

// ---- block state changes -----------------------------------------------------
// Remove a resident block from the pool (eviction or invalidation); returns
// its group.  Callers account the per-group statistics, warp-aggregated.
// clear_res: also clear the resident bit (evictions leave it: the id is
// allocated again in the same step, and k_bm_write sets the allocated bits).
__device__ uint32_t drop_block(const DevState& s, uint32_t b, bool clear_res = true) {
  table_delete(s, b);
  const uint32_t g = s.blk_group[b];
  s.blk_flags[b] = 0;
  if (clear_res) atomicAnd(s.res_bits + (b >> 5), ~(1u << (b & 31)));
  return g;
}

// Position -> (request, position within the request).
struct PosRef {
  uint32_t i;
  int m;
};
__device__ __forceinline__ bool pos_ref(const DevState& s, int64_t pos, PosRef* r) {
  if (pos >= s.ctl->nblocks) return false;
  r->i = s.pos_req[pos];  // both loads in one round trip
  r->m = (int)s.pos_m[pos];
  return true;
}

// ===========================================================================
// Init: an empty pool, every balance at beta (Sec. III-B, B = beta at t = 0).
__global__ void k_init_blocks(DevState s) {
  const int64_t nclaims = (int64_t)kClaimWays << s.cl_nbuckets_log2;
  for (int64_t c = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; c < nclaims; c += (int64_t)gridDim.x * blockDim.x) {
    s.claims[c] = empty_claim();
  }
}
__global__ void k_init_ctl(DevState s) {
  if (threadIdx.x == 0 && blockIdx.x == 0) {
    Ctl c{};
    c.step = 1;
    c.stamp_base = 1;
    *s.ctl = c;
  }
  for (int i = threadIdx.x; i < s.G * s.C; i += blockDim.x) s.ledger[i] = s.beta[i % s.C];
}

// ===========================================================================
// Stage 0: validation of the step's inputs; n_i, block positions and the
// chunk descriptors of the hashing stage.  One CTA per kValTile requests;
// the exclusive scans of blocks and chunks over the requests take each
// tile's base from its predecessors' published totals (a decoupled look-back
// without inclusive prefixes: a tile sums every earlier tile's total, and no
// total waits on anything).  The last CTA to finish sets the call's status
// and per-step scalars, and clears the tile words for the next call.
// 'probe' skips the clock and step checks.  Every write is bounds-checked, so
// inputs that turn out invalid write nothing outside the scratch arrays.
constexpr uint64_t kTileFlag = 1ull << 63;

__global__ void __launch_bounds__(kValTile) k_validate(DevState s, int probe) {
  s = with_args(s);
  __shared__ uint64_t s_base;
  __shared__ bool s_last;
  Ctl* c = s.ctl;
  const int R = s.R;
  const int tile = blockIdx.x;
  const int i = tile * kValTile + (int)threadIdx.x;
  const bool in = i < R;
  bool bad = false;
  int32_t n = 0, ns = 0, cid = 0, g = 0;
  int64_t o0 = 0;
  if (in) {
    o0 = s.in_offsets[i];
    const int64_t o1 = s.in_offsets[i + 1];
    g = s.in_group[i];
    const int64_t nb = (o1 - o0) / s.bs;
    bad = o1 < o0 || g < 0 || g >= s.G || nb > (int64_t)kMaxPos;
    if (s.in_contract) {
      cid = s.in_contract[i];
      bad |= cid < 0 || cid >= s.C;
    } else if (!probe && !bad) {
      cid = s.contract_of_group[g];
    }
    if (s.in_prefix) bad |= s.in_prefix[i] == 0;
    n = bad ? 0 : (int32_t)nb;
  }
  ns = (n + kChunkBlocks - 1) / kChunkBlocks;
  const int tile_bad = __syncthreads_or(bad);
  // blocks in the high half, chunks in the low half of one scanned word
  uint64_t tot;
  const uint64_t ex = block_excl_scan<uint64_t>((uint64_t)n << 32 | (uint64_t)ns, &tot);
  if (threadIdx.x == 0) st_relaxed_u64(s.val_tile + tile, tot | kTileFlag);
  if (threadIdx.x < 32 && tile * kValTile < R) {  // the tile's base: every earlier tile's total
    const int lane = threadIdx.x;
    uint64_t sum = 0;
    bool ok = true;
    for (int t0 = 0; t0 < tile; t0 += 32) {
      if (t0 + lane < tile) {
        const uint64_t v = wait_word(s.val_tile + t0 + lane, kTileFlag);
        ok = ok && v != 0;
        sum += v & ~kTileFlag;
      }
    }
    sum = warp_sum(sum);
    if (!__all_sync(kFull, ok) && lane == 0) atomicOr(&c->v_bad, 2u);  // never expected
    if (lane == 0) s_base = sum;
  } else if (threadIdx.x == 0) {
    s_base = 0;  // a tile past the step's requests writes nothing
  }
  __syncthreads();
  const uint64_t e = s_base + ex;
  const int64_t pbase = (int64_t)(e >> 32), sbase = (int64_t)(uint32_t)e;
  if (in && pbase + n <= s.max_blocks && sbase + ns <= s.max_segments) {
    s.rq_n[i] = n;
    s.rq_h[i] = n;
    s.rq_s[i] = n;
    s.rq_fu[i] = kNone;
    s.rq_pbase[i] = (int32_t)pbase;
    if (!probe) {
      s.rq_cid[i] = cid;
      s.rq_hs[i] = kNone;  // a request with no full block has no history entry
      s.rq_p[i] = 0;
    }
  }
  // each request's chunk descriptors; the warp writes one request's chunks
  // at a time, so the stores coalesce
  const bool room = in && pbase + n <= s.max_blocks && sbase + ns <= s.max_segments;
  for (unsigned todo = __ballot_sync(kFull, room && ns > 0); todo; todo &= todo - 1) {
    const int src = __ffs(todo) - 1;
    const int64_t ro0 = __shfl_sync(kFull, o0, src);
    const int64_t rsb = __shfl_sync(kFull, sbase, src);
    const int32_t rpb = (int32_t)__shfl_sync(kFull, pbase, src);
    const int32_t rn = __shfl_sync(kFull, n, src), rns = __shfl_sync(kFull, ns, src);
    const uint32_t ri = (uint32_t)__shfl_sync(kFull, i, src), rg = (uint32_t)__shfl_sync(kFull, g, src);
    for (int k = lane_id(); k < rns; k += 32) {
      ChunkDesc d;
      d.o0 = ro0;
      d.req = ri;
      d.n = rn;
      d.pbase = rpb;
      d.k = k;
      d.group = rg;
      d.sb = (int32_t)rsb;
      s.chunks[rsb + k] = d;
      s.seg_word[rsb + k] = 0;
    }
  }
  if (!probe && tile == 0) {  // per-step counts accumulated by later kernels
    if (s.policy == PS_STATICQUOTA)
      for (int gg = threadIdx.x; gg < s.G; gg += blockDim.x) s.grp_pinned[gg] = 0;
    for (int r = threadIdx.x; r < s.G * kClasses; r += blockDim.x) {  // the candidate counts (k_cand)
      if (r < s.G) s.grp_qsize[r] = 0;
      s.cls[r] = ClsRange{0, ~0u, 0, ~0u, 0};
    }
  }
  // the last CTA to finish: status and per-call scalars
  if (threadIdx.x == 0) {
    if (tile_bad) atomicOr(&c->v_bad, 1u);
    if (tot) atomicAdd(reinterpret_cast<unsigned long long*>(&c->v_sum), (unsigned long long)tot);
    __threadfence();
    s_last = atomicAdd(&c->v_ticket, 1u) == gridDim.x - 1;
  }
  __syncthreads();
  if (!s_last) return;
  __threadfence();
  for (int t = threadIdx.x; t < (int)gridDim.x; t += blockDim.x) s.val_tile[t] = 0;
  if (threadIdx.x != 0) return;
  // every value the verdict needs, loaded up front so the loads overlap
  const uint32_t vb = ldcg_u32(&c->v_bad);
  const uint64_t all = ldcg_u64(&c->v_sum);  // blocks (high half) and chunks (low half) of the step
  const int64_t T = R > 0 ? s.in_offsets[R] : 0;
  const int64_t first_off = R > 0 ? s.in_offsets[0] : 0;
  const int32_t sticky = c->sticky;
  const int64_t t_prev = c->t_prev;
  const uint64_t step = c->step;
  c->v_bad = 0;
  c->v_ticket = 0;
  c->v_sum = 0;
  int32_t st = PS_OK;
  if (!probe && sticky != PS_OK) st = sticky;
  else if (!probe && s.now < t_prev) st = PS_ERR_CLOCK;
  else if (!probe && step > kMaxStep) st = PS_ERR_CAPACITY;
  else if (vb || first_off != 0 || T > s.max_tokens) st = PS_ERR_INVALID_ARG;
  c->status = st;
  c->T = T;
  c->hash_ticket = 0;
  if (st != PS_OK) {
    c->nblocks = 0;
    c->nsegs = 0;
    return;
  }
  c->nblocks = (int64_t)(all >> 32);
  c->nsegs = (int64_t)(uint32_t)all;
  if (!probe) {
    c->pinned = 0; c->n_inval = 0; c->total_claims = 0; c->avail = 0; c->need = 0;
    c->nfree = 0; c->ftake = 0; c->mvict = 0; c->hist_new = 0; c->n_evicted = 0;
    c->n_alloc = 0; c->n_victims_marked = 0; c->m_fb = 0; c->sel_ntie = 0; c->sel_k = 0; c->ticket = 0;
    c->internal_error = (vb & 2) ? 1 : 0;
    c->nlaunch = 1;  // this kernel; every later kernel of the step adds itself
  }
}

// ===========================================================================
// Stages 1-2 in one kernel: chained block hashing (Sec. III-B native content
// key), the longest cached prefix (n_cached of Alg. 1), the pins of the
// cached prefix, the claims of every block past it, and each request's
// history entry (OnRequest of Alg. 1).
//
// A chunk is up to kChunkBlocks = 64 consecutive blocks of one prompt; one
// warp takes one chunk, lane l its blocks l and 32 + l (two halves).  Chunks
// are numbered in request order (a request's chunks are consecutive) and CTAs
// draw their chunks in that order from a ticket, so every chunk's
// predecessors belong to warps that have already started.  Each lane reads
// its blocks' tokens with 16-byte loads and forms the block digests D_m
// itself.  The chain C_m = Kc C_{m-1} + D_m (mod 2^61 - 1) composes affine
// maps, so a warp scan of each half gives each block its chain value B_m
// relative to the half's start (value 0 entering it); the chunk's total, the
// second half's total plus Kc^(its blocks) times the first's, is published
// under a flag.  (Two blocks a lane halve the chunks, and with them the
// chain of dependent accesses each one pays: ticket, descriptor,
// predecessors' totals and miss bits.)  The value entering chunk k of a
// request is then
//   Kc^(64k) C_seed + sum_{l<k} Kc^(64(k-1-l)) total_l,
// and no total waits on anything, so the warp folds its k predecessors'
// totals directly, in windows of 32 (one lane each).  With C_m the lanes form
// their keys and probe the table.  A block is in the cached prefix iff no
// block before it in its request misses: the chunk's "some block missed" bit
// is the second published flag, and the warp ORs its predecessors'.  The
// cached prefix is pinned for the step; every block past it is claimed in the
// claim map (lowest request index wins: one materialization, one charge, I1).
// The warp of a request's first chunk installs the request's history entry.
//
// Each chunk publishes one 64-bit word (seg_word, zeroed per call by
// k_validate): bits 0-60 its chain total (a value mod 2^61 - 1), bit 61 set
// once the total is there, bit 62 once its miss bit (bit 63) is.  Value and
// flags travel in one aligned 64-bit store, read with one relaxed 64-bit
// load, so no fence orders them.  Every wait is bounded; a wait that runs
// out reports an internal error.
constexpr uint64_t kWordTotal = 1ull << 61, kWordMiss = 1ull << 62, kWordMissBit = 1ull << 63;
// A chunk descriptor in two 16-byte loads.
__device__ __forceinline__ ChunkDesc load_chunk(const ChunkDesc* p) {
  const uint4 a = __ldg(reinterpret_cast<const uint4*>(p)), b = __ldg(reinterpret_cast<const uint4*>(p) + 1);
  ChunkDesc d;
  d.o0 = (int64_t)((uint64_t)a.y << 32 | a.x);
  d.req = a.z;
  d.n = (int32_t)a.w;
  d.pbase = (int32_t)b.x;
  d.k = (int32_t)b.y;
  d.group = b.z;
  d.sb = (int32_t)b.w;
  return d;
}

// NH sums over a piece of PIECE tokens held in w[] from word OFF on (OFF the
// warp-uniform word offset, a compile-time constant in each of four forms),
// with key words from pair index kk0 on.  Summing straight from w[] keeps
// no second, re-indexed copy of the tokens live.
template <int OFF, int PIECE, int NWORDS>
__device__ __forceinline__ void nh_piece(const uint32_t (&w)[NWORDS], const uint32_t* sk, int kk0, uint64_t* a1,
                                         uint64_t* a2) {
#pragma unroll
  for (int k = 0; k < PIECE / 2; ++k) {
    const int kk = kk0 + k;
    const uint32_t tx = w[OFF + 2 * k], ty = w[OFF + 2 * k + 1];
    *a1 += (uint64_t)(tx + sk[2 * kk]) * (uint64_t)(ty + sk[2 * kk + 1]);
    *a2 += (uint64_t)(tx + sk[2 * kk + 2]) * (uint64_t)(ty + sk[2 * kk + 3]);
  }
}

// The two NH sums of one block (bs tokens from token index g0).  r is the
// request's word offset (g0 mod 4, the same for all its blocks); with a
// 16-byte aligned token buffer the block's tokens are read as the 16-byte
// words that cover them, 16 tokens at a time, otherwise token by token (as
// they are near the step's last token, where the covering words could pass
// it).
template <int BS>
__device__ __forceinline__ void block_nh(const DevState& s, const uint32_t* sk, int64_t g0, int r, bool vec, int64_t T,
                                         uint64_t* d1, uint64_t* d2) {
  constexpr int PIECE = BS < 16 ? BS : 16;  // tokens per piece
  uint64_t a1 = 0, a2 = 0;
#pragma unroll
  for (int q0 = 0; q0 < BS; q0 += PIECE) {
    const int64_t a0 = g0 + q0 - r;
    bool done = false;
    if constexpr (PIECE % 4 == 0) {
      constexpr int NW = PIECE / 4 + 1;  // 16-byte words covering a piece at any word offset
      if (vec && a0 + 4 * NW <= T) {
        uint32_t w[4 * NW];
        const uint4* src = reinterpret_cast<const uint4*>(s.in_tokens + a0);
#pragma unroll
        for (int q = 0; q < NW; ++q) {
          const uint4 v = __ldg(src + q);
          w[4 * q] = v.x;
          w[4 * q + 1] = v.y;
          w[4 * q + 2] = v.z;
          w[4 * q + 3] = v.w;
        }
        switch (r) {  // warp-uniform
          case 0: nh_piece<0, PIECE>(w, sk, q0 / 2, &a1, &a2); break;
          case 1: nh_piece<1, PIECE>(w, sk, q0 / 2, &a1, &a2); break;
          case 2: nh_piece<2, PIECE>(w, sk, q0 / 2, &a1, &a2); break;
          default: nh_piece<3, PIECE>(w, sk, q0 / 2, &a1, &a2); break;
        }
        done = true;
      }
    }
    if (!done) {
      uint32_t w[PIECE];
#pragma unroll
      for (int j = 0; j < PIECE; ++j) w[j] = (uint32_t)s.in_tokens[g0 + q0 + j];
      nh_piece<0, PIECE>(w, sk, q0 / 2, &a1, &a2);
    }
  }
  *d1 = a1;
  *d2 = a2;
}

// One chunk (j) of k_hash_lookup, by one warp.  Returns false if a wait for
// a predecessor ran out (never expected).
template <int BS>
__device__ __forceinline__ bool hash_lookup_chunk(const DevState& s, Ctl* c, const uint32_t* sk, const uint64_t* kc,
                                                  int64_t j, int probe) {
  const int lane = lane_id();
  const ChunkDesc d = load_chunk(s.chunks + j);
  const uint32_t i = d.req;
  const int n = d.n;
  const int64_t sb = d.sb;
  const int k = d.k;  // chunk index within the request
  const int m0 = k * kChunkBlocks;
  const int nb = tmin(kChunkBlocks, n - m0);
  const int nbA = tmin(kSegBlocks, nb), nbB = nb - nbA;  // blocks of the two halves
  const int64_t o0 = d.o0;
  const int pbase = d.pbase;
  const uint32_t g = d.group;
  const int64_t T = c->T;
  const int mA = m0 + lane, mB = m0 + kSegBlocks + lane;
  // D_m of the lane's two blocks, then the inclusive scans of the affine maps
  // x -> Kc x + D, one per half
  uint64_t bA = 0, bB = 0;
  if (lane < nbA) {
    uint64_t d1, d2;
    block_nh<BS>(s, sk, o0 + (int64_t)mA * BS, (int)(o0 & 3), s.tokens_aligned16 != 0, T, &d1, &d2);
    bA = add61(red61(d1), mul61(s.digest_mul, red61(d2)));
  }
  if (lane < nbB) {
    uint64_t d1, d2;
    block_nh<BS>(s, sk, o0 + (int64_t)mB * BS, (int)(o0 & 3), s.tokens_aligned16 != 0, T, &d1, &d2);
    bB = add61(red61(d1), mul61(s.digest_mul, red61(d2)));
  }
#pragma unroll
  for (int q = 0; q < 5; ++q) {
    const uint64_t tA = __shfl_up_sync(kFull, bA, 1 << q);
    const uint64_t tB = __shfl_up_sync(kFull, bB, 1 << q);
    if (lane >= (1 << q)) {
      bA = add61(bA, mul61(kc[1 << q], tA));
      bB = add61(bB, mul61(kc[1 << q], tB));
    }
  }
  const uint64_t totA = __shfl_sync(kFull, bA, nbA - 1);
  const uint64_t totB = __shfl_sync(kFull, bB, nbB > 0 ? nbB - 1 : 0);
  // a second half follows a full first half (Kc^32 times it)
  const uint64_t total = nbB > 0 ? add61(mul61(kc[nbB], totA), totB) : totA;
  if (lane == 0) st_relaxed_u64(s.seg_word + j, total | kWordTotal);
  // the chain value entering the chunk
  bool ok = true;
  uint64_t cin = red61(chain_seed(s.hash_seed, (int32_t)g));
  for (int l0 = 0; l0 < k; l0 += 32) {
    const int w = tmin(32, k - l0);
    uint64_t term = 0;
    if (lane < w) {
      const uint64_t v = wait_word(s.seg_word + sb + l0 + lane, kWordTotal);
      ok = ok && v != 0;
      term = mul61(kc[(kSegBlocks + 1) + (w - 1 - lane)], v & kP61);
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) term = add61(term, __shfl_xor_sync(kFull, term, o));
    cin = add61(mul61(kc[(kSegBlocks + 1) + w], cin), term);
  }
  // the lane's keys and their table probes
  uint64_t keyA = 0, keyB = 0;
  uint32_t blkA = kNone, blkB = kNone;
  if (lane < nbA) {
    const uint64_t C = add61(mul61(kc[lane + 1], cin), bA);
    keyA = fix_reserved(mix64(C ^ ((uint64_t)(mA + 1) * 0xD1B54A32D192ED03ull)));
  }
  if (lane < nbB) {
    const uint64_t cinB = add61(mul61(kc[kSegBlocks], cin), totA);
    const uint64_t C = add61(mul61(kc[lane + 1], cinB), bB);
    keyB = fix_reserved(mix64(C ^ ((uint64_t)(mB + 1) * 0xD1B54A32D192ED03ull)));
  }
  if (lane < nbA) blkA = table_find(s, keyA, g);
  if (lane < nbB) blkB = table_find(s, keyB, g);
  const unsigned missA = __ballot_sync(kFull, lane < nbA && blkA == kNone);
  const unsigned missB = __ballot_sync(kFull, lane < nbB && blkB == kNone);
  const bool anymiss = (missA | missB) != 0;
  if (lane == 0) st_relaxed_u64(s.seg_word + j, total | kWordTotal | kWordMiss | (anymiss ? kWordMissBit : 0));
  // did any earlier block of the request miss?
  bool missbefore = false;
  for (int l0 = 0; l0 < k && !missbefore; l0 += 32) {
    const int w = tmin(32, k - l0);
    bool mb = false;
    if (lane < w) {
      const uint64_t v = wait_word(s.seg_word + sb + l0 + lane, kWordMiss);
      ok = ok && v != 0;
      mb = (v & kWordMissBit) != 0;
    }
    missbefore = __any_sync(kFull, mb);
  }
  if (!__all_sync(kFull, ok)) return false;  // a predecessor never published
  // first miss in this chunk
  const int first = missA ? __ffs(missA) - 1 : (missB ? kSegBlocks + __ffs(missB) - 1 : kChunkBlocks);
  if (!missbefore && anymiss && lane == 0) s.rq_h[i] = m0 + first;  // h_i: its only writer
  if (probe) return true;
  const uint32_t step32 = (uint32_t)c->step;
  // the cached prefix is pinned, every later block claimed
  auto place = [&](bool act, int half, uint64_t key, uint32_t blk, uint32_t* klass) -> bool {
    if (!act) return false;
    const int mm = m0 + half * kSegBlocks + lane;
    const int64_t p = pbase + mm;
    s.pos_key[p] = key;
    s.pos_req[p] = i;
    s.pos_m[p] = (uint32_t)mm;
    s.pos_blk[p] = blk;
    bool pinned = false;
    if (!missbefore && half * kSegBlocks + lane < first) {
      pinned = atomicExch(s.blk_pin + blk, step32) != step32;
      if (pinned && s.lg_on) *klass = s.blk_klass[blk];
      s.pos_claim[p] = kNone;
    } else {
      s.pos_claim[p] = claim_insert(s, key, i);
    }
    return pinned;
  };
  uint32_t klassA = 0, klassB = 0;
  const bool pinA = place(lane < nbA, 0, keyA, blkA, &klassA);
  const bool pinB = place(lane < nbB, 1, keyB, blkB, &klassB);
  const int np = __popc(__ballot_sync(kFull, pinA)) + __popc(__ballot_sync(kFull, pinB));
  if (lane == 0 && np) atomic_add_i64(&c->pinned, np);
  // hits are namespaced by group: every block the warp pins is group g's
  if (s.policy == PS_STATICQUOTA && lane == 0 && np) atomic_add_i64(s.grp_pinned + g, np);
  if (s.lg_on) {  // a pinned block is no candidate: it leaves its queues' live counts (applied in k_lg_cand)
    const int32_t A1 = lg_log_a(s, g, klassA), B1 = lg_log_b(s, klassA);
    agg_add_i64(s.lg_pin, (uint32_t)A1, 1, pinA && A1 >= 0);
    agg_add_i64(s.lg_pin, (uint32_t)B1, 1, pinA && B1 >= 0);
    const int32_t A2 = lg_log_a(s, g, klassB), B2 = lg_log_b(s, klassB);
    agg_add_i64(s.lg_pin, (uint32_t)A2, 1, pinB && A2 >= 0);
    agg_add_i64(s.lg_pin, (uint32_t)B2, 1, pinB && B2 >= 0);
  }
  const uint64_t key = keyA;  // block 0's key, in the first chunk's lane 0
  // OnRequest of Alg. 1: the request's (group, prefix) history entry
  if (k == 0 && lane == 0) {
    const uint64_t pid = s.in_prefix ? s.in_prefix[i] : key;  // default: block 0's key
    uint32_t hs = kNone;
    const uint32_t hmask = (1u << s.hist_cap_log2) - 1;
    uint32_t x = hist_home(pid, g, s.hist_cap_log2);
    for (uint32_t it = 0; it <= hmask; ++it, x = (x + 1) & hmask) {
      uint64_t olo, ohi;
      cas128(s.hist + x, 0ull, 0ull, pid, (uint64_t)(g + 1), &olo, &ohi);
      if (olo == 0 && ohi == 0) {
        atomic_add_i64(&c->hist_new, 1);
        hs = x;
        break;
      }
      if (olo == pid && (uint32_t)ohi == g + 1) {
        hs = x;
        break;
      }
    }
    if (hs != kNone)
      atomicMax(reinterpret_cast<unsigned long long*>(&s.hist[hs].ftag), (unsigned long long)step_tag(c->step, i));
    s.rq_hs[i] = hs;
    s.rq_p[i] = pid;
  }
  return true;
}

// The kernel: persistent warps.  Each warp takes chunk tickets one at a time,
// each only once it is free to start the chunk, so a chunk's predecessors
// (lower tickets) have always started hashing before it, and their totals
// arrive about when its own does.  A chunk waits only on chunks of lower
// tickets, each held by a running warp: the waits always make progress.
// probe = 1: the read-only probe (ps_cached_prefix): h_i only, no pins,
// claims, history or per-position records.
constexpr int kHashCtasPerSm = 5;
template <int BS>
__global__ void __launch_bounds__(256, kHashCtasPerSm) k_hash_lookup(DevState s, int probe) {
  s = with_args(s);
  __shared__ uint32_t sk[BS + 2];                // the NH key words (read by every lane alike)
  __shared__ uint64_t kc[2 * (kSegBlocks + 1)];  // Kc^j, then Kc^(32 t)
  Ctl* c = s.ctl;
  if (c->status != PS_OK) return;
  if (threadIdx.x < BS + 2) sk[threadIdx.x] = s.key_words[threadIdx.x];
  if (threadIdx.x < 2 * (kSegBlocks + 1)) kc[threadIdx.x] = s.kc_pow[threadIdx.x];
  __syncthreads();
  const int lane = lane_id();
  const int64_t nsegs = c->nsegs;
  for (;;) {
    uint32_t t = 0;
    if (lane == 0) t = atomicAdd(&c->hash_ticket, 1u);
    t = __shfl_sync(kFull, t, 0);
    if ((int64_t)t >= nsegs) return;
    if (!hash_lookup_chunk<BS>(s, c, sk, kc, (int64_t)t, probe)) {
      if (lane == 0) c->internal_error = 1;
      return;
    }
  }
}


// A step whose new (group, prefix) entries would overflow the history map
// fails as a whole, leaving the pool as it was (Alg. 1's hooks change state
// only for a request that goes ahead).  k_hash_lookup has written three things
// by then, undone here thread by thread over the same positions and requests:
//  - pin tags of the cached prefix: set to a tag no step compares against
//    (the previous step's), so the retried step pins them afresh;
//  - claim-map entries: cleared (the map holds only this step's keys);
//  - history entries: an entry with no committed reference was installed by
//    this step and is removed (entries are never removed otherwise, so no
//    probe sequence ran through it); every other touched entry loses the
//    step's first-reference tag.
// The error itself is raised by k_grant, after every thread here is done.
__device__ __forceinline__ bool history_overflows(const DevState& s, const Ctl* c) {
  return c->hist_live + c->hist_new > s.history_capacity;
}
__device__ void undo_pin_claim(const DevState& s, const Ctl* c, int64_t t) {
  const int64_t nb = c->nblocks;
  const uint32_t step32 = (uint32_t)c->step;
  if (t < nb) {
    PosRef r;
    pos_ref(s, t, &r);
    if (r.m < s.rq_h[r.i]) {
      s.blk_pin[s.pos_blk[t]] = step32 - 1u;
    } else {
      const uint32_t slot = s.pos_claim[t];
      if (slot != kNone) s.claims[slot] = empty_claim();
    }
  } else if (t < nb + s.R) {
    const uint32_t hs = s.rq_hs[t - nb];
    if (hs != kNone) {
      HistEntry* e = s.hist + hs;
      if (ldcg_u32(&e->refadm) == 0) *e = HistEntry{};
      else e->ftag = 0;
    }
  }
}

// A history entry from L2 (two 16-byte loads that skip L1: a tag may have
// been updated by an atomic since another CTA on this SM read the line).
__device__ __forceinline__ HistEntry ldcg_hist(const HistEntry* p) {
  const uint4 a = __ldcg(reinterpret_cast<const uint4*>(p)), b = __ldcg(reinterpret_cast<const uint4*>(p) + 1);
  HistEntry e;
  e.p = (uint64_t)a.y << 32 | a.x;
  e.g1 = a.z;
  e.refadm = a.w;
  e.ftag = (uint64_t)b.y << 32 | b.x;
  e.atag = (uint64_t)b.w << 32 | b.z;
  return e;
}

// Stage 2 (cont.): the first own claim s_i of each request, and orphans.  A
// resident block past a request's first miss cannot be reached by lookup; it
// is dropped (invalidated) unless some request pinned it.  Threads past the
// positions take the requests (used only to undo a failing step).
__global__ void __launch_bounds__(kThreads) k_claims(DevState s) {
  s = with_args(s);
  Ctl* c = s.ctl;
  if (c->status != PS_OK) return;
  if (history_overflows(s, c)) {
    undo_pin_claim(s, c, blockIdx.x * (int64_t)blockDim.x + threadIdx.x);
    return;
  }
  const int64_t pos = blockIdx.x * (int64_t)blockDim.x + threadIdx.x;
  const uint32_t step32 = (uint32_t)c->step;
  bool inv = false;
  uint32_t ginv = 0, kinv = 0;
  PosRef r;
  bool own = false;
  const bool valid = pos_ref(s, pos, &r);
  if (valid) {
    const int h = s.rq_h[r.i];
    own = r.m >= h && ldcg_u32(&s.claims[s.pos_claim[pos]].minreq) == r.i;
    if (r.m > h) {
      const uint32_t b = s.pos_blk[pos];
      if (b != kNone && ldcg_u32(s.blk_pin + b) != step32 && atomicExch(s.blk_inval + b, step32) != step32) {
        ginv = drop_block(s, b);
        if (s.lg_on) kinv = s.blk_klass[b];
        atomicOr(s.bm_inval + (b >> 5), 1u << (b & 31));
        inv = true;
      }
    }
  }
  // s_i = the first own claim: one atomic per request per warp
  agg_min_u32(reinterpret_cast<uint32_t*>(s.rq_s), valid ? r.i : 0u, valid ? (uint32_t)r.m : 0u, own);
  if (s.lg_on) {  // an invalidated block leaves its queues
    const int32_t A = lg_log_a(s, ginv, kinv), B = lg_log_b(s, kinv);
    agg_add_i64(s.lg_live, (uint32_t)A, -1, inv && A >= 0);
    agg_add_i64(s.lg_live, (uint32_t)B, -1, inv && B >= 0);
  }
  agg_stat(s, ginv, PS_STAT_INVALIDATED_BLOCKS, 1, inv);
  agg_stat(s, ginv, PS_STAT_RESIDENT_BLOCKS, -1, inv);
  const int ni = __popc(__ballot_sync(kFull, inv));
  if (lane_id() == 0 && ni) {
    atomic_add_i64(&c->n_inval, ni);
    atomic_add_i64(&c->n_resident, -ni);
  }
}

// ===========================================================================
// Stage 3: grant new blocks against the pool.  avail = free + unpinned
// resident = N - pinned; claims are ranked in (request, position) order; the
// first avail ranks are materialized.  One CTA.
__global__ void __launch_bounds__(1024) k_grant(DevState s0) {
  // Contract arrays are read from the parameter block: indexing the per-step
  // copy by a run-time contract would move the whole copy to local memory.
  const DevState s = with_args(s0);
  extern __shared__ unsigned long long g_sum[];  // [G * C] the step's charges per (group, contract)
  Ctl* c = s.ctl;
  if (c->status != PS_OK) return;
  if (history_overflows(s, c)) {  // undone by k_claims; the error is sticky
    if (threadIdx.x == 0) { c->status = PS_ERR_CAPACITY; c->sticky = PS_ERR_CAPACITY; }
    return;
  }
  const int R = s.R;
  const int C = s.C;
  const bool quota = s.policy == PS_STATICQUOTA;  // a_i already granted per group
  for (int k = threadIdx.x; k < s.G * C; k += blockDim.x) g_sum[k] = 0;
  __syncthreads();
  const int64_t avail = s.N - c->pinned;
  // Granted ranks are the first avail in (request, position) order, so the
  // grants before request i number min(avail, base_i), base_i the claims
  // before it, and a_i = min(avail, base_i + c_i) - min(avail, base_i).  One
  // scanned word per request: claims in the high half, StaticQuota grants in
  // the low; four 1024-request sub-tiles a pass.
  uint64_t carry = 0;
  const int tile = 4 * (int)blockDim.x;
  for (int t0 = 0; t0 < R; t0 += tile) {
    uint64_t v[4], ex[4];
    int32_t cl[4], aq[4];
#pragma unroll
    for (int u = 0; u < 4; ++u) {
      const int i = t0 + u * (int)blockDim.x + (int)threadIdx.x;
      const bool in = i < R;
      cl[u] = in ? s.rq_n[i] - s.rq_s[i] : 0;
      aq[u] = in && quota ? s.rq_a[i] : 0;
      v[u] = (uint64_t)cl[u] << 32 | (uint64_t)aq[u];
    }
    uint64_t tot;
    block_excl_scan4(v, ex, &tot);
#pragma unroll
    for (int u = 0; u < 4; ++u) {
      const int i = t0 + u * (int)blockDim.x + (int)threadIdx.x;
      if (i < R) {
        const uint64_t e = carry + ex[u];
        const int64_t base_c = (int64_t)(e >> 32);
        const int64_t lo = quota ? (int64_t)(uint32_t)e : tmin(avail, base_c);
        const int32_t a = quota ? aq[u] : (int32_t)(tmin(avail, base_c + cl[u]) - lo);
        // granted keys are paired with the allocated ids in (request,
        // position) order: request i's first granted key is the lo-th
        s.rq_cbase[i] = (int32_t)lo;
        s.rq_a[i] = a;
        s.out.admitted_blocks[i] = a;
        s.out.admitted_offsets[i] = (int32_t)lo;
        if (a > 0) atomicAdd(&g_sum[s.in_group[i] * C + s.rq_cid[i]], (unsigned long long)a);
      }
    }
    carry += tot;
  }
  const int64_t carry_c = (int64_t)(carry >> 32);
  const int64_t carry_a = quota ? (int64_t)(uint32_t)carry : tmin(avail, carry_c);
  int64_t qv = 0;  // StaticQuota: the groups' overflows are the victims
  if (quota)
    for (int g = threadIdx.x; g < s.G; g += blockDim.x) qv += s.grp_x[g];
  qv = block_sum(qv);
  if (threadIdx.x == 0) {
    const int64_t need = carry_a;
    s.out.admitted_offsets[R] = (int32_t)need;
    const int64_t nfree = s.N - c->n_resident;
    c->avail = avail;
    c->total_claims = carry_c;
    c->need = need;
    c->nfree = nfree;
    c->ftake = quota ? need - qv : tmin(need, nfree);
    c->mvict = need - c->ftake;
  }
  // The step's balances and debts (Eq. 1-3, 5) follow from each (group,
  // contract)'s total charge, so they are settled here and the select need
  // not wait for the per-request metering (which reads the refilled opening
  // balances from ledger_b0).
  __syncthreads();
  const int64_t unit = (int64_t)1 << s.fp_shift;
  for (int g = threadIdx.x; g < s.G; g += blockDim.x) {
    int64_t raw = 0, norm = 0, rmax = 0;
    for (int cc = 0; cc < C; ++cc) {
      const int64_t b0 = refill(s.ledger[g * C + cc], s0.beta[cc], s0.rho[cc], s.now - c->t_prev);
      s.ledger_b0[g * C + cc] = b0;
      const int64_t b = b0 - (int64_t)g_sum[g * C + cc] * unit;  // Eq. 2 over the step's charges
      s.ledger[g * C + cc] = b;
      const int64_t def = tmax<int64_t>(0, -b);
      raw += def;                                    // Eq. 3
      norm += muldiv(def, s.rho_min, s0.rho[cc]);    // Eq. 5
      if (b < 0) rmax = tmax(rmax, s0.rho[cc]);
    }
    int64_t* row = s.stats + (int64_t)g * PS_NUM_STATS;
    row[PS_STAT_DEBT_RAW] = raw;
    row[PS_STAT_DEBT_NORM] = norm;
    s.out.debt_raw[g] = raw;
    s.out.debt_norm[g] = norm;
    s.grp_P[g] = norm;
    s.grp_delta[g] = rmax ? muldiv(unit, s.rho_min, rmax) : 0;  // 1/W_g of Eq. 8
    SelSeg z{};
    z.kmin = ~0ull;
    z.kmax = 0;
    z.qmin = ~0ull;
    z.qmax = 0;
    s.sel[g] = z;
  }
}

// StaticQuota (Sec. V-A) grants, one CTA per group: the group's claims, in
// (request, position) order, while its partition of Q = floor(N / G) blocks
// minus its pinned ones holds them; its overflow m_g = granted - (Q -
// resident) is what it must reclaim from its own blocks.
__global__ void __launch_bounds__(1024) k_grant_quota(DevState s) {
  s = with_args(s);
  Ctl* c = s.ctl;
  if (c->status != PS_OK) return;
  const int g = blockIdx.x;
  const int64_t Q = s.N / s.G;
  const int64_t avail = Q - s.grp_pinned[g];
  const int R = s.R;
  int64_t carry = 0, granted = 0;
  for (int t0 = 0; t0 < R; t0 += blockDim.x) {
    const int i = t0 + threadIdx.x;
    const bool member = i < R && s.in_group[i] == g;
    const int32_t cl = member ? s.rq_n[i] - s.rq_s[i] : 0;
    int32_t tot;
    const int32_t ex = block_excl_scan(cl, &tot);
    if (member) {
      const int64_t a = tmin<int64_t>(cl, tmax<int64_t>(0, avail - (carry + ex)));
      s.rq_a[i] = (int32_t)a;
      granted += a;
    }
    carry += tot;
  }
  granted = block_sum(granted);
  if (threadIdx.x == 0) {
    const int64_t resident = s.stats[(int64_t)g * PS_NUM_STATS + PS_STAT_RESIDENT_BLOCKS];
    s.grp_x[g] = tmax<int64_t>(0, granted - (Q - resident));
  }
}

// In-step hits: positions of [h_i, s_i) belong to earlier requests' claims;
// the leading granted ones are hits.  A position whose owner's key was not
// granted lowers the request's first-ungranted mark.
__global__ void __launch_bounds__(kThreads) k_instep(DevState s) {
  s = with_args(s);
  const Ctl* c = s.ctl;
  if (c->status != PS_OK) return;
  const int64_t pos = blockIdx.x * (int64_t)blockDim.x + threadIdx.x;
  PosRef r;
  bool past = false;
  const bool valid = pos_ref(s, pos, &r);
  if (valid && r.m >= s.rq_h[r.i] && r.m < s.rq_s[r.i]) {
    // the owner's claims are ranked consecutively: its key here is granted
    // iff it is among the owner's first a_j
    const uint32_t j = s.claims[s.pos_claim[pos]].minreq;
    past = r.m - s.rq_s[j] >= s.rq_a[j];
  }
  agg_min_u32(s.rq_fu, valid ? r.i : 0u, valid ? (uint32_t)r.m : 0u, past);
}

// ===========================================================================
// Stages 3-4: metering (Eq. 1-3, OnCacheFullBlocks of Alg. 1), in request
// order, one CTA per group.  The CTA compacts its group's requests of each
// tile of kMeterTile requests into shared memory (in request order), then
// works on the members only: block-wide exclusive scans give each member the
// charges of the group's earlier requests per contract, hence
//   D_g before the request (the gate of OnTouch, Eq. 4),
//   B_{g,c} after the request's own charge (the class of its new blocks).
// q_r >= 1 and "(g,p) was admitted" come from the history entry as it stood at
// the start of the step and the first request of the step that referenced /
// admitted it.  Also writes the group's request statistics; the balances
// and debts after the step are k_grant's (from the same charges).
constexpr int kMeterThreads = 512;
constexpr int kMeterTile = 4 * kMeterThreads;  // requests compacted per pass
__global__ void __launch_bounds__(kMeterThreads) k_meter(DevState s0) {
  // Contract arrays are read from the parameter block: indexing the per-step
  // copy by a run-time contract would move the whole copy to local memory.
  const DevState s = with_args(s0);
  Ctl* c = s.ctl;
  if (c->status != PS_OK) return;
  const int g = blockIdx.x;
  const int C = s.C;
  const int64_t unit = (int64_t)1 << s.fp_shift;
  const uint64_t step = c->step;
  __shared__ int64_t B0[PS_MAX_CONTRACTS];
  __shared__ unsigned long long s_st[7];  // the group's request statistics
  __shared__ int32_t s_mem[kMeterTile];   // this tile's members, in request order
  if (threadIdx.x < C) B0[threadIdx.x] = s.ledger_b0[g * C + threadIdx.x];  // refilled by k_grant
  if (threadIdx.x < 7) s_st[threadIdx.x] = 0;
  __syncthreads();
  int64_t carry[PS_MAX_CONTRACTS];
#pragma unroll
  for (int cc = 0; cc < PS_MAX_CONTRACTS; ++cc) carry[cc] = 0;
  int64_t st_req = 0, st_ptok = 0, st_full = 0, st_hit = 0, st_inst = 0, st_adm = 0, st_ungr = 0;
  const int R = s.R;
  for (int base = 0; base < R; base += kMeterTile) {
    // members of this tile: four consecutive requests a thread, compacted by
    // a block scan of their counts (the order is request order)
    const int i0 = base + 4 * (int)threadIdx.x;
    int32_t gg[4] = {-1, -1, -1, -1};
    if (i0 + 3 < R && (reinterpret_cast<uintptr_t>(s.in_group + i0) & 15) == 0) {
      const int4 v = *reinterpret_cast<const int4*>(s.in_group + i0);
      gg[0] = v.x; gg[1] = v.y; gg[2] = v.z; gg[3] = v.w;
    } else {
#pragma unroll
      for (int u = 0; u < 4; ++u)
        if (i0 + u < R) gg[u] = s.in_group[i0 + u];
    }
    int cnt = 0;
#pragma unroll
    for (int u = 0; u < 4; ++u) cnt += gg[u] == g;
    int nmem;
    int at = block_excl_scan(cnt, &nmem);
#pragma unroll
    for (int u = 0; u < 4; ++u)
      if (gg[u] == g) s_mem[at++] = i0 + u;
    __syncthreads();
    for (int k0 = 0; k0 < nmem; k0 += kMeterThreads) {
      const int k = k0 + (int)threadIdx.x;
      const bool mem = k < nmem;
      const int i = mem ? s_mem[k] : 0;
      int n = 0, a = 0, cid = 0, rh = 0, re = 0, rs = 0;
      uint32_t hs = kNone, fu = kNone;
      int64_t ptok = 0;
      if (mem) {
        n = s.rq_n[i]; a = s.rq_a[i]; cid = s.rq_cid[i]; hs = s.rq_hs[i];
        rh = s.rq_h[i]; rs = s.rq_s[i]; fu = s.rq_fu[i];
        ptok = s.in_offsets[i + 1] - s.in_offsets[i];
        // in-step hits: the leading positions of [h_i, s_i) before the first
        // ungranted one; hit_i = h_i + e_i
        re = (int)tmin<uint32_t>(fu, (uint32_t)rs) - rh;
        s.rq_e[i] = re;
        s.out.hit_blocks[i] = rh + re;
        // the first admitting request of the (group, prefix) entry in this
        // step: only requests of this group share its entries, and every one
        // of them is this CTA's
        if (a > 0 && hs != kNone)
          atomicMax(reinterpret_cast<unsigned long long*>(&s.hist[hs].atag), (unsigned long long)step_tag(step, (uint32_t)i));
      }
      const bool pol = mem && n > 0;
      __syncthreads();  // every member's admission tag is in place
      HistEntry he{};
      if (pol && hs != kNone) he = ldcg_hist(s.hist + hs);
      // charges of this group's earlier requests, per contract
      int64_t S[PS_MAX_CONTRACTS];
#pragma unroll
      for (int cc = 0; cc < PS_MAX_CONTRACTS; ++cc) {
        S[cc] = 0;
        if (cc < C) {
          int64_t tot;
          const int64_t ex = block_excl_scan<int64_t>((pol && cid == cc) ? a : 0, &tot);
          S[cc] = carry[cc] + ex;
          carry[cc] += tot;
        }
      }
      if (pol) {
        // the raw debt before this request's charge (Eq. 3) and its balance after
        int64_t d = 0, b_after = 0;
#pragma unroll
        for (int cc = 0; cc < PS_MAX_CONTRACTS; ++cc) {
          if (cc < C) {
            d += tmax<int64_t>(0, -(B0[cc] - S[cc] * unit));
            if (cid == cc) b_after = B0[cc] - (S[cc] + a) * unit;
          }
        }
        const bool gate = (s.flags & PS_FLAG_NO_DEBT_GATE) || d <= s.eps;
        const uint32_t refadm = he.refadm;
        const bool q_ge1 = (refadm & 0x7FFFFFFFu) >= 1 || tag_req(he.ftag, step) < (uint32_t)i;
        const bool adm_before = (refadm >> 31) || tag_req(he.atag, step) < (uint32_t)i;
        const bool proven = q_ge1 && adm_before;
        s.rq_flags[i] = (uint8_t)((proven ? 1 : 0) | (gate ? 2 : 0));
        s.rq_knew[i] = (uint8_t)((b_after < -s.eps || !adm_before) ? kProb : kNormal);
        st_full += n; st_hit += rh + re; st_inst += re; st_adm += a; st_ungr += (n - rs) - a;
      }
      if (mem) { st_req += 1; st_ptok += ptok; }
    }
    __syncthreads();  // s_mem is rewritten by the next tile
  }
  {
    const int64_t v[7] = {st_req, st_ptok, st_full, st_hit, st_inst, st_adm, st_ungr};
#pragma unroll
    for (int k = 0; k < 7; ++k) {
      const int64_t w = warp_sum(v[k]);
      if (lane_id() == 0 && w) atomicAdd(&s_st[k], (unsigned long long)w);
    }
  }
  __syncthreads();
  st_req = (int64_t)s_st[0]; st_ptok = (int64_t)s_st[1]; st_full = (int64_t)s_st[2]; st_hit = (int64_t)s_st[3];
  st_inst = (int64_t)s_st[4]; st_adm = (int64_t)s_st[5]; st_ungr = (int64_t)s_st[6];
  if (threadIdx.x == 0) {
    int64_t* row = s.stats + (int64_t)g * PS_NUM_STATS;
    row[PS_STAT_REQUESTS] += st_req;
    row[PS_STAT_PROMPT_TOKENS] += st_ptok;
    row[PS_STAT_FULL_BLOCKS] += st_full;
    row[PS_STAT_HIT_BLOCKS] += st_hit;
    row[PS_STAT_INSTEP_HIT_BLOCKS] += st_inst;
    row[PS_STAT_HIT_TOKENS] += st_hit * s.bs;
    row[PS_STAT_ADMITTED_BLOCKS] += st_adm;
    row[PS_STAT_UNGRANTED_BLOCKS] += st_ungr;
  }
}

// ===========================================================================
// Stage 4: OnTouch (Alg. 1, Eq. 4) for every hit block, resident or in-step,
// thread per position.  Pass 1 applies the access updates (stamp = max,
// access count, S3-FIFO frequency) and records, per block, the lowest request
// whose touch promotes it.  Pass 2 counts the gated touches that precede the
// promotion (or all of them when none promotes) and applies the promotion of
// resident blocks.
__global__ void __launch_bounds__(kThreads) k_touch(DevState s) {
  s = with_args(s);
  const Ctl* c = s.ctl;
  if (c->status != PS_OK) return;
  const int64_t pos = blockIdx.x * (int64_t)blockDim.x + threadIdx.x;
  PosRef r;
  if (!pos_ref(s, pos, &r)) return;
  const uint32_t i = r.i;
  const int m = r.m;
  const int h = s.rq_h[i];
  if (m >= h + s.rq_e[i]) return;
  const uint8_t fl = s.rq_flags[i];
  const bool proven = fl & 1, gate = fl & 2;
  const int cid = s.rq_cid[i];
  const uint64_t p = s.rq_p[i];
  const uint64_t step = c->step;
  bool elig;
  if (m < h) {
    const uint32_t b = s.pos_blk[pos];
    atomicMax(reinterpret_cast<unsigned long long*>(s.blk_stamp + b),
              (unsigned long long)make_stamp(c->stamp_base, s.rq_pbase[i], s.rq_n[i], m));
    if (s.lg_on) s.lg_slot[s.rq_pbase[i] + (s.rq_n[i] - 1 - m)] = b;  // the queues' append reads it back
    atomicAdd(s.blk_acc + b, 1u);
    atomicAdd(s.blk_freq + b, 1u);
    elig = proven && s.blk_contract[b] == cid && s.blk_prefix[b] == p && s.blk_klass[b] != kReuse;
    if (elig && gate)
      atomicMax(reinterpret_cast<unsigned long long*>(s.blk_promo + b), (unsigned long long)step_tag(step, i));
  } else {
    ClaimEntry* e = s.claims + s.pos_claim[pos];
    const uint32_t j = e->minreq;
    // later requests give larger stamps: the maximum is the latest touch's
    atomicMax(reinterpret_cast<unsigned long long*>(&e->stamp),
              (unsigned long long)make_stamp(c->stamp_base, s.rq_pbase[i], s.rq_n[i], m));
    atomicAdd(&e->tcnt, 1u);
    elig = proven && s.rq_cid[j] == cid && s.rq_p[j] == p;  // new blocks are never Reuse yet
    if (elig && gate) atomicMin(&e->promo, i);
  }
  s.pos_elig[pos] = elig;
}

__global__ void __launch_bounds__(kThreads) k_touch2(DevState s) {
  s = with_args(s);
  const Ctl* c = s.ctl;
  if (c->status != PS_OK) return;
  const int64_t pos = blockIdx.x * (int64_t)blockDim.x + threadIdx.x;
  PosRef r;
  int gated = 0, promoted = 0;
  uint32_t g = 0;
  if (pos_ref(s, pos, &r) && r.m < s.rq_h[r.i] + s.rq_e[r.i] && s.pos_elig[pos]) {
    const uint32_t i = r.i;
    g = (uint32_t)s.in_group[i];
    const bool gate = s.rq_flags[i] & 2;
    uint32_t promoter, b = kNone;
    if (r.m < s.rq_h[i]) {
      b = s.pos_blk[pos];
      promoter = tag_req(ldcg_u64(s.blk_promo + b), c->step);
    } else {
      promoter = ldcg_u32(&s.claims[s.pos_claim[pos]].promo);
    }
    if (!gate) {
      gated = i < promoter;
    } else if (i == promoter) {
      promoted = 1;
      if (b != kNone) s.blk_klass[b] = kReuse;
    }
  }
  agg_stat(s, g, PS_STAT_GATED_REUSES, gated, gated != 0);
  agg_stat(s, g, PS_STAT_PROMOTIONS, promoted, promoted != 0);
}

// ===========================================================================
// Stage 5: reclamation.  Candidates are resident blocks not hit in this step.
// The order key is (class, stamp) for prefixshield (Eq. 9; stamp only with
// the no-segmentation ablation) and the stamp for lru.  Per (segment, class):
// the candidates and their stamp range, so the radix select can start inside
// the class that holds its rank and skip the bytes the class's stamps share.
__global__ void __launch_bounds__(1024) k_cand(DevState s) {
  s = with_args(s);
  extern __shared__ uint32_t cand_smem[];  // 5 arrays of nseg * kClasses
  Ctl* c = s.ctl;
  if (c->status != PS_OK) return;  // runs beside S3-S4: the victim count is not known yet
  const uint32_t step32 = (uint32_t)c->step;
  // segments: groups for prefixshield and staticquota, one for lru; retention
  // classes only for prefixshield
  const bool ps = s.policy == PS_PREFIXSHIELD || s.policy == PS_STATICQUOTA;
  const bool seg = s.policy == PS_PREFIXSHIELD && !(s.flags & PS_FLAG_NO_SEGMENTATION);
  const int nrow = (ps ? s.G : 1) * kClasses;
  uint32_t* s_cnt = cand_smem;
  uint32_t* s_hmin = s_cnt + nrow;
  uint32_t* s_hmax = s_hmin + nrow;
  uint32_t* s_lmin = s_hmax + nrow;
  uint32_t* s_lmax = s_lmin + nrow;
  for (int r = threadIdx.x; r < nrow; r += blockDim.x) {
    s_cnt[r] = 0;
    s_hmin[r] = s_lmin[r] = ~0u;
    s_hmax[r] = s_lmax[r] = 0;
  }
  __syncthreads();
  // kU blocks a thread per iteration, their loads issued together; the trip
  // count is warp-uniform.  Lanes of one (segment, class) combine their
  // ranges and counts with warp reductions; one lane updates shared memory.
  constexpr int kU = 4;
  const int64_t span = (int64_t)gridDim.x * blockDim.x;
  for (int64_t b0 = blockIdx.x * (int64_t)blockDim.x; b0 < s.N; b0 += span * kU) {
    uint8_t fl[kU], kl[kU];
    uint32_t pin[kU];
    uint16_t grp[kU];
    uint64_t st[kU];
#pragma unroll
    for (int u = 0; u < kU; ++u) {
      const int64_t b = b0 + u * span + threadIdx.x;
      fl[u] = 0;
      if (b < s.N) {
        fl[u] = s.blk_flags[b];
        kl[u] = s.blk_klass[b];
        pin[u] = s.blk_pin[b];
        grp[u] = s.blk_group[b];
        st[u] = s.blk_stamp[b];
      }
    }
#pragma unroll
    for (int u = 0; u < kU; ++u) {
      const int64_t b = b0 + u * span + threadIdx.x;
      uint64_t key = ~0ull;
      uint32_t row = ~0u;
      if ((fl[u] & 1) && pin[u] != step32) {
        key = seg ? (st[u] | (uint64_t)kl[u] << 62) : st[u];
        row = (ps ? (uint32_t)grp[u] : 0u) * kClasses + (seg ? kl[u] : 0u);
      }
      const unsigned peers = __match_any_sync(kFull, row);
      if (row != ~0u) {
        const uint32_t hi = (uint32_t)(st[u] >> 32), lo = (uint32_t)st[u];
        const uint32_t hmin = __reduce_min_sync(peers, hi), hmax = __reduce_max_sync(peers, hi);
        const uint32_t lmin = __reduce_min_sync(peers, lo), lmax = __reduce_max_sync(peers, lo);
        if (lane_id() == __ffs(peers) - 1) {
          atomicAdd(&s_cnt[row], (unsigned)__popc(peers));
          atomicMin(&s_hmin[row], hmin);
          atomicMax(&s_hmax[row], hmax);
          atomicMin(&s_lmin[row], lmin);
          atomicMax(&s_lmax[row], lmax);
        }
      }
      if (b < s.N) s.csk[b] = key;
    }
  }
  __syncthreads();
  for (int r = threadIdx.x; r < nrow; r += blockDim.x) {
    if (!s_cnt[r]) continue;
    if (ps) atomic_add_i64(s.grp_qsize + r / kClasses, s_cnt[r]);
    ClsRange* d = s.cls + r;
    atomicAdd(&d->cnt, s_cnt[r]);
    atomicMin(&d->hmin, s_hmin[r]);
    atomicMax(&d->hmax, s_hmax[r]);
    atomicMin(&d->lmin, s_lmin[r]);
    atomicMax(&d->lmax, s_lmax[r]);
  }
}

// Stamp range of a class from its two half ranges: exact below the top half
// when every member shares its top 32 bits, conservative otherwise.
__device__ __forceinline__ void cls_stamp_range(const ClsRange& r, uint64_t* lo, uint64_t* hi) {
  const bool same_hi = r.hmin == r.hmax;
  *lo = ((uint64_t)r.hmin << 32) | (same_hi ? r.lmin : 0u);
  *hi = ((uint64_t)r.hmax << 32) | (same_hi ? r.lmax : 0xFFFFFFFFu);
}

__device__ __forceinline__ void sel_start(SelSeg& z);
// Start a segment's search from its per-class candidates: the class holding
// the rank-th smallest key is fixed (lower classes are all below it), the rank
// becomes a rank inside that class, and the key range is the class's.
// cnt[k] and [lo[k], hi[k]] describe class k (unsegmented keys: class 0 only).
// Classes are picked without run-time array indexing (registers only).
__device__ __forceinline__ void sel_start_cls(SelSeg& z, const int64_t (&cnt)[kClasses], const uint64_t (&lo)[kClasses],
                                              const uint64_t (&hi)[kClasses], bool segmented) {
  static_assert(kClasses == 3, "class choice below is written for three classes");
  int k = 0;
  int64_t below = 0;
  if (segmented && z.rank > cnt[0]) {
    below = cnt[0];
    k = 1;
    if (z.rank > cnt[0] + cnt[1]) {
      below += cnt[1];
      k = 2;
    }
  }
  const int64_t ck = k == 0 ? cnt[0] : k == 1 ? cnt[1] : cnt[2];
  const uint64_t lk = k == 0 ? lo[0] : k == 1 ? lo[1] : lo[2];
  const uint64_t hk = k == 0 ? hi[0] : k == 1 ? hi[1] : hi[2];
  const uint64_t cb = segmented ? (uint64_t)k << 62 : 0ull;
  if (z.active && ck > 0) {
    z.rank -= below;
    z.kmin = cb | lk;
    z.kmax = cb | hk;
  } else {
    z.kmin = z.kmax = cb;
  }
  sel_start(z);
}
__device__ __forceinline__ void sel_start_group(const DevState& s, int g, SelSeg& z, bool segmented) {
  int64_t cnt[kClasses];
  uint64_t lo[kClasses], hi[kClasses];
#pragma unroll
  for (int k = 0; k < kClasses; ++k) {
    const ClsRange r = s.cls[g * kClasses + k];
    cnt[k] = r.cnt;
    cls_stamp_range(r, &lo[k], &hi[k]);
  }
  sel_start_cls(z, cnt, lo, hi, segmented);
}

// One global segment: all candidates for lru, or (fallback) the candidates
// the debt phase of prefixshield left, in (class, stamp) order (Eq. 9).  The
// debt phase took group g's x_g smallest keys, so of class k it took
// clamp(x_g - (members of lower classes), 0, members of class k).
// One warp: the segment-0 state of a global select (lru, or the fallback).
__device__ void start_global_select(const DevState& s, Ctl* c, int fallback) {
  const int lane = lane_id();
  int64_t m = 0;
  if (c->status == PS_OK) m = fallback ? c->m_fb : c->mvict;
  const bool segmented = s.policy == PS_PREFIXSHIELD && !(s.flags & PS_FLAG_NO_SEGMENTATION);
  int64_t cnt[kClasses];
  uint64_t lo[kClasses], hi[kClasses];
  for (int k = 0; k < kClasses; ++k) { cnt[k] = 0; lo[k] = ~0ull; hi[k] = 0; }
  if (m > 0) {
    const int nseg = fallback ? s.G : 1;
    for (int g = lane; g < nseg; g += 32) {
      int64_t taken = fallback ? s.grp_x[g] : 0;
      for (int k = 0; k < kClasses; ++k) {
        const ClsRange r = s.cls[g * kClasses + k];
        const int64_t t = tmin<int64_t>(taken, (int64_t)r.cnt);
        taken -= t;
        if ((int64_t)r.cnt > t) {
          uint64_t a, b;
          cls_stamp_range(r, &a, &b);
          cnt[k] += (int64_t)r.cnt - t;
          lo[k] = tmin(lo[k], a);
          hi[k] = tmax(hi[k], b);
        }
      }
    }
    for (int k = 0; k < kClasses; ++k)
      for (int o = 16; o > 0; o >>= 1) {
        cnt[k] += __shfl_xor_sync(kFull, cnt[k], o);
        lo[k] = tmin(lo[k], (uint64_t)__shfl_xor_sync(kFull, lo[k], o));
        hi[k] = tmax(hi[k], (uint64_t)__shfl_xor_sync(kFull, hi[k], o));
      }
  }
  if (lane != 0) return;
  SelSeg z{};
  z.rank = m;
  z.active = m > 0;
  z.incl = 1;
  z.qmin = ~0ull;
  z.qmax = 0;
  sel_start_cls(z, cnt, lo, hi, segmented);
  s.sel[0] = z;
  c->lst_n = 0;
}
__global__ void __launch_bounds__(32) k_sel_single(DevState s, int fallback) {
  s = with_args(s);
  start_global_select(s, s.ctl, fallback);
}

// StaticQuota: each group reclaims its overflow m_g from its own blocks, in
// recency order (one segment per group, no global fallback).
__global__ void __launch_bounds__(1024) k_quota_sel(DevState s) {
  s = with_args(s);
  Ctl* c = s.ctl;
  const int64_t m = c->status == PS_OK ? c->mvict : 0;
  for (int g = threadIdx.x; g < s.G; g += blockDim.x) {
    SelSeg z = s.sel[g];
    z.rank = m > 0 ? s.grp_x[g] : 0;
    z.active = z.rank > 0;
    z.incl = 1;
    sel_start_group(s, g, z, false);
    s.sel[g] = z;
  }
  if (threadIdx.x == 0) { c->m_fb = 0; c->sel_ntie = 0; c->sel_k = 0; c->lst_n = 0; }
}

// Alg. 2 in closed form (one CTA).  Group g's j-th victim would be taken at
// projected value v_{g,j} = P_g - j*delta_g (Eq. 8) while v_{g,j} > epsilon
// (Eq. 6); each group's sequence strictly decreases, so the per-victim argmax
// loop (Eq. 7) takes items in order of (value descending, candidate key
// ascending).  The m-th largest value tau splits the items: every item above
// tau is taken; among the groups holding an item at exactly tau (at most one
// each) the ones with the smallest candidate keys are taken (resolved after
// the radix select finds those keys).  What the debt phase cannot cover goes
// to the global fallback in (class, stamp) order.
__global__ void __launch_bounds__(1024) k_waterfill(DevState s, cudaGraphConditionalHandle fb_cond, int has_cond) {
  s = with_args(s);
  Ctl* c = s.ctl;
  __shared__ int64_t sP[PS_MAX_GROUPS], sD[PS_MAX_GROUPS], sQ[PS_MAX_GROUPS];
  __shared__ uint64_t sRcp[PS_MAX_GROUPS];  // floor((2^64 - 1) / d) for the division below
  __shared__ int64_t s_pmax;
  const int G = s.G;
  const int64_t eps = s.eps;
  const bool seg = !(s.flags & PS_FLAG_NO_SEGMENTATION);
  const int64_t m = (c->status == PS_OK) ? c->mvict : 0;
  if (m == 0) {
    for (int g = threadIdx.x; g < G; g += blockDim.x) { s.sel[g].active = 0; s.grp_x[g] = 0; s.grp_full[g] = 0; }
    if (threadIdx.x == 0) c->m_fb = 0;
    return;
  }
  for (int g = threadIdx.x; g < G; g += blockDim.x) {
    sP[g] = s.grp_P[g];
    sD[g] = s.grp_delta[g];
    sQ[g] = s.grp_qsize[g];
    sRcp[g] = sD[g] > 1 ? ~0ull / (uint64_t)sD[g] : 0;
  }
  if (threadIdx.x == 0) s_pmax = 0;
  __syncthreads();
  // floor(x / d) for x >= 0 from the reciprocal: the estimate is at most two
  // below the quotient, and the correction makes it exact
  auto div_d = [&](int g, uint64_t x) -> uint64_t {
    const uint64_t d = (uint64_t)sD[g];
    if (d == 1) return x;
    uint64_t q = __umul64hi(x, sRcp[g]);
    while (x - q * d >= d) ++q;
    return q;
  };
  // items of group g with value > t: min(q, floor((P - t - 1) / d) + 1) if P > t
  auto items_gt = [&](int g, int64_t t) -> int64_t {
    const int64_t P = sP[g], d = sD[g];
    return (P > t && d > 0) ? tmin<int64_t>(sQ[g], (int64_t)div_d(g, (uint64_t)(P - t - 1)) + 1) : 0;
  };
  int64_t e = 0, pm = 0;
  for (int g = threadIdx.x; g < G; g += blockDim.x) { e += items_gt(g, eps); pm = tmax(pm, sP[g]); }
  const int64_t E = block_sum(e);
  if (pm) atomicMax(reinterpret_cast<unsigned long long*>(&s_pmax), (unsigned long long)pm);
  __syncthreads();
  if (E <= m) {
    // a group that gives all its candidates needs no select: the split takes
    // them whole
    for (int g = threadIdx.x; g < G; g += blockDim.x) {
      const int64_t x = items_gt(g, eps);
      const bool full = x > 0 && x == sQ[g];
      s.grp_x[g] = x;
      s.grp_full[g] = full ? 1 : 0;
      SelSeg z = s.sel[g];
      z.rank = full ? 0 : x;
      z.active = x > 0 && !full;
      z.incl = 1;
      sel_start_group(s, g, z, seg);
      s.sel[g] = z;
    }
    if (threadIdx.x == 0) {
      c->m_fb = m - E; c->sel_ntie = 0; c->sel_k = 0; c->lst_n = 0;
      if (has_cond && m > E) cudaGraphSetConditional(fb_cond, 1);  // the queues' fallback phase runs
    }
    return;
  }
  // tau = max{t in [eps+1, pmax] : items_gt(t - 1) summed >= m}.  Only the
  // groups that can hold an item above eps count (d > 0, q > 0, P > eps);
  // each round tests T thresholds spread over the interval, L lanes (a power
  // of two covering them, at most 32) splitting the groups of one: each
  // evaluation is a chain of dependent 64-bit steps, so one per thread and
  // more rounds beat several per thread and fewer rounds.
  __shared__ int16_t s_gid[PS_MAX_GROUPS];
  __shared__ int s_ng;
  __shared__ int s_J[3];
  {
    int k = 0;
    for (int base = 0; base < G; base += blockDim.x) {
      const int g = base + threadIdx.x;
      const bool holds = g < G && sD[g] > 0 && sQ[g] > 0 && sP[g] > eps;
      int tot;
      const int ex = block_excl_scan((int)holds, &tot);
      if (holds) s_gid[k + ex] = (int16_t)g;
      k += tot;
    }
    if (threadIdx.x == 0) s_ng = k;
    if (threadIdx.x < 3) s_J[threadIdx.x] = -1;
    __syncthreads();
  }
  const int ng = s_ng;
  int64_t lo = eps + 1, hi = s_pmax;
  {
    int L = 1, logT = 10;  // blockDim.x == 1024 == T * L
    while (L < ng && L < 32) { L <<= 1; --logT; }
    const int T = 1 << logT;
    const int jt = threadIdx.x / L, gl = threadIdx.x % L;
    for (int r = 0; lo < hi; ++r) {
      const int64_t span = hi - lo;  // >= 1
      const int64_t stride = tmax<int64_t>(1, (span + T - 1) >> logT);
      auto thr = [&](int jj) -> int64_t { return jj == T - 1 ? hi : tmin<int64_t>(hi, lo + 1 + stride * jj); };
      const int64_t t = thr(jt);
      int64_t cnt = 0;
      for (int k = gl; k < ng; k += L) cnt += items_gt(s_gid[k], t - 1);
      for (int o = L / 2; o > 0; o >>= 1) cnt += __shfl_xor_sync(kFull, cnt, o);
      // J = the largest threshold still holding m items (counts fall as the
      // threshold rises); slots rotate over three rounds, so one barrier a
      // round separates every slot's reset, updates and reads
      if (threadIdx.x == 0) s_J[(r + 1) % 3] = -1;
      if (gl == 0 && cnt >= m) atomicMax(&s_J[r % 3], jt);
      __syncthreads();
      const int J = s_J[r % 3];
      if (J < 0) {
        hi = lo;
      } else {
        // both ends from this round's lo (thr reads lo and hi by reference)
        const int64_t nlo = thr(J), nhi = J + 1 < T ? thr(J + 1) - 1 : hi;
        lo = nlo;
        hi = nhi < nlo ? nlo : nhi;
      }
    }
  }
  const int64_t tau = lo;
  int64_t above = 0, ntie = 0;
  for (int g = threadIdx.x; g < G; g += blockDim.x) {
    const int64_t P = sP[g], d = sD[g], q = sQ[g];
    const int64_t xa = items_gt(g, tau);
    const uint64_t qt = (d > 0 && P >= tau) ? div_d(g, (uint64_t)(P - tau)) : 0;
    const bool tied = d > 0 && P >= tau && qt * (uint64_t)d == (uint64_t)(P - tau) && (int64_t)qt < q;
    above += xa;
    ntie += tied;
    SelSeg z = s.sel[g];
    z.rank = xa + (tied ? 1 : 0);
    z.active = z.rank > 0;
    z.incl = tied ? 2 : 1;  // 2: the tie item is taken only if the tie rule chooses it
    sel_start_group(s, g, z, seg);
    s.sel[g] = z;
    s.grp_x[g] = xa + (tied ? 1 : 0);
    s.grp_full[g] = 0;
  }
  above = block_sum(above);
  ntie = block_sum(ntie);
  if (threadIdx.x == 0) {
    c->m_fb = 0;
    c->lst_n = 0;
    c->sel_ntie = (int32_t)ntie;
    c->sel_k = (int32_t)(m - above);  // tied items to take, 1..ntie
  }
}

// ---- exact segmented select -------------------------------------------------
// Each active segment (a group in the debt phase, one global segment for lru
// and for the fallback) looks for the rank-th smallest key among its
// candidates, MSB-first, one byte at a time.  Bytes that all its candidates
// share (from their smallest and largest key) are fixed without counting.
// The first counted byte is histogrammed over the whole candidate array;
// a split pass then marks every candidate below the chosen bucket as a
// victim and copies the bucket's members into a short list, over which the
// remaining bytes are counted.  A last-CTA-done resolve picks each digit.

// Highest byte where kmin and kmax differ, as a shift; -1 if equal.
__device__ __forceinline__ int first_shift(uint64_t kmin, uint64_t kmax) {
  const uint64_t d = kmin ^ kmax;
  return d == 0 ? -1 : ((63 - __clzll((long long)d)) / 8) * 8;
}
// Bytes above 'shift' (shift a multiple of 8 in [0, 56]).
__device__ __forceinline__ uint64_t above_mask(int shift) { return shift >= 56 ? 0ull : (~0ull << (shift + 8)); }
// The next unresolved digit under a byte-aligned prefix mask, or -1.
__device__ __forceinline__ int next_shift(uint64_t mask) {
  if (mask == ~0ull) return -1;
  if (mask == 0) return 56;
  return __ffsll((long long)mask) - 1 - 8;
}
// Start a segment's search from its key range (rank and activity already set).
__device__ __forceinline__ void sel_start(SelSeg& z) {
  const int fs = first_shift(z.kmin, z.kmax);
  if (fs < 0) {
    z.prefix = z.kmin;
    z.mask = ~0ull;
  } else {
    z.mask = above_mask(fs);
    z.prefix = z.kmin & z.mask;
  }
}

// A segment as the list passes see it: the list's members of the segment all
// share the bits above the highest byte where the list's smallest and largest
// key differ, so those bytes are fixed without counting.
__device__ __forceinline__ SelSeg list_view(SelSeg z) {
  if (z.qmin > z.qmax) return z;  // no member on the list
  const int fs = first_shift(z.qmin, z.qmax);
  const uint64_t cm = fs < 0 ? ~0ull : above_mask(fs);
  z.mask |= cm;
  z.prefix |= z.qmin & cm;
  return z;
}

// The first counted digit of every segment, over the whole candidate array:
// 16 bits wide (two bytes) while at most kWideRows segments count, one byte
// otherwise, into global histograms (warp-aggregated atomics).  CTA 0 records
// the rows' segments for k_wide_resolve.
__device__ __forceinline__ void wide_digit(int nrows, uint64_t mask, int* dshift, uint32_t* nbins) {
  const int sh = next_shift(mask);
  const bool w16 = nrows <= kWideRows && sh >= 8;
  *dshift = w16 ? sh - 8 : sh;
  *nbins = w16 ? (uint32_t)kWideBins : (uint32_t)kRadixBins;
}
__global__ void __launch_bounds__(256) k_wide_pass(DevState s, int single, int fallback) {
  s = with_args(s);
  __shared__ uint32_t s_coarse[kRadixBins];  // one row's coarse counts (a single segment)
  __shared__ int16_t row_of[PS_MAX_GROUPS];
  __shared__ uint64_t s_pre[PS_MAX_GROUPS], s_msk[PS_MAX_GROUPS];  // the segments' prefix and mask
  __shared__ int s_nrows;
  Ctl* c = s.ctl;
  if (c->status != PS_OK || c->mvict == 0) return;
  const int nseg = single ? 1 : s.G;
  if (single && !s.sel[0].active) return;
  {
    int k = 0;
    for (int base = 0; base < nseg; base += blockDim.x) {
      const int g = base + threadIdx.x;
      bool counts = false;
      if (g < nseg) {
        const SelSeg ss = s.sel[g];
        counts = ss.active && next_shift(ss.mask) >= 0;
        s_pre[g] = ss.prefix;
        s_msk[g] = ss.mask;
      }
      int tot;
      const int ex = block_excl_scan((int)counts, &tot);
      if (g < nseg) row_of[g] = counts ? (int16_t)(k + ex) : (int16_t)-1;
      if (counts && blockIdx.x == 0) s.wide_seg[k + ex] = (int16_t)g;
      k += tot;
    }
    if (threadIdx.x == 0) {
      s_nrows = k;
      if (blockIdx.x == 0) c->wide_nrows = k;
    }
    __syncthreads();
  }
  const int nrows = s_nrows;
  if (nrows == 0) return;
  const uint32_t stride = nrows <= kWideRows ? (uint32_t)kWideBins : (uint32_t)kRadixBins;
  // A 16-bit digit is also counted by its top byte (row-major, 256 a row)
  // for the resolve.  One row takes every candidate (lru, the fallback):
  // its 256 coarse counts would serialize global atomics, so each CTA counts
  // them in shared memory and adds its nonzero ones once at the end.
  const bool coarse_smem = nrows == 1 && stride == (uint32_t)kWideBins;
  for (int k = threadIdx.x; k < kRadixBins; k += blockDim.x) s_coarse[k] = 0;
  __syncthreads();
  // kU candidates a thread per iteration, their loads issued together (the
  // trip count is CTA-uniform, as the warp-aggregated increment needs)
  constexpr int kU = 4;
  const int64_t span = (int64_t)gridDim.x * blockDim.x;
  for (int64_t b0 = blockIdx.x * (int64_t)blockDim.x; b0 < s.N; b0 += span * kU) {
    uint64_t key[kU];
    int seg[kU];
    uint32_t vw[kU];
#pragma unroll
    for (int u = 0; u < kU; ++u) {
      const int64_t e = b0 + u * span + threadIdx.x;
      key[u] = ~0ull;
      seg[u] = 0;
      vw[u] = 0;
      if (e < s.N) {
        key[u] = s.csk[e];
        if (!single) seg[u] = s.blk_group[e];
        if (fallback) vw[u] = s.bm_victim[e >> 5];
      }
    }
#pragma unroll
    for (int u = 0; u < kU; ++u) {
      const int64_t e = b0 + u * span + threadIdx.x;
      bool act = false, act16 = false;
      uint32_t idx = 0;
      if (key[u] != ~0ull && !((vw[u] >> (e & 31)) & 1)) {
        const int row = row_of[seg[u]];
        if (row >= 0) {
          const uint64_t msk = s_msk[seg[u]];
          if ((key[u] & msk) == s_pre[seg[u]]) {
            int dsh;
            uint32_t nb;
            wide_digit(nrows, msk, &dsh, &nb);
            act = true;
            act16 = nb == (uint32_t)kWideBins;
            idx = (uint32_t)row * stride + (uint32_t)((key[u] >> dsh) & (nb - 1));
          }
        }
      }
      agg_inc(s.wide_bins, idx, act);
      const uint32_t cidx = (idx >> 16) * kRadixBins + ((idx >> 8) & 0xFF);
      if (coarse_smem) {
        if (act16) atomicAdd(&s_coarse[cidx], 1u);
      } else if (stride == (uint32_t)kWideBins) {
        agg_inc(s.wide_coarse, cidx, act16);
      }
    }
  }
  if (coarse_smem) {
    __syncthreads();
    for (int k = threadIdx.x; k < kRadixBins; k += blockDim.x)
      if (s_coarse[k]) atomicAdd(s.wide_coarse + k, s_coarse[k]);
  }
}

// One warp per counted segment: the bucket holding the segment's rank-th key
// fixes the digit.  A 16-bit digit is found in two short scans (its top byte
// from the coarse histogram, then the 256 bins under it); the coarse bins are
// cleared here and the fine ones by the split that follows.
__global__ void __launch_bounds__(32) k_wide_resolve(DevState s, int single) {
  s = with_args(s);
  Ctl* c = s.ctl;
  if (c->status != PS_OK || c->mvict == 0) return;
  if (single && !s.sel[0].active) return;
  const int nrows = c->wide_nrows;
  const int r = blockIdx.x;
  if (r >= nrows) return;
  const int lane = lane_id();
  const int seg = s.wide_seg[r];
  SelSeg ss = s.sel[seg];
  int dsh;
  uint32_t nb;
  wide_digit(nrows, ss.mask, &dsh, &nb);
  const bool w16 = nb == (uint32_t)kWideBins;
  const uint32_t stride = nrows <= kWideRows ? (uint32_t)kWideBins : (uint32_t)kRadixBins;
  uint32_t* row = s.wide_bins + (size_t)r * stride;
  // locate rank among 256 consecutive bins (8 a lane); returns the bin and
  // the count before it
  auto locate = [&](const uint32_t* bins, uint64_t rank, uint32_t* before) -> uint32_t {
    uint32_t v[8], sum = 0;
#pragma unroll
    for (int k = 0; k < 8; ++k) { v[k] = __ldcg(bins + lane * 8 + k); sum += v[k]; }
    const uint32_t incl = warp_incl_scan(sum), excl = incl - sum;
    const bool mine = (uint64_t)excl < rank && rank <= (uint64_t)incl;
    const unsigned mw = __ballot_sync(kFull, mine);
    const int ml = mw ? __ffs(mw) - 1 : 0;
    uint32_t d = 0, run = excl;
    if (mine) {
      for (int k = 0; k < 8; ++k) {
        if (rank <= (uint64_t)(run + v[k])) { d = lane * 8 + k; break; }
        run += v[k];
      }
    }
    *before = __shfl_sync(kFull, run, ml);
    return __shfl_sync(kFull, d, ml);
  };
  uint32_t d, run;
  if (w16) {
    uint32_t* coarse = s.wide_coarse + (size_t)r * kRadixBins;
    uint32_t cb_before;
    const uint32_t cb = locate(coarse, (uint64_t)ss.rank, &cb_before);
    uint32_t fb_before;
    const uint32_t fb = locate(row + cb * kRadixBins, (uint64_t)ss.rank - cb_before, &fb_before);
    d = cb * kRadixBins + fb;
    run = cb_before + fb_before;
#pragma unroll
    for (int k = 0; k < 8; ++k) coarse[lane * 8 + k] = 0;
  } else {
    d = locate(row, (uint64_t)ss.rank, &run);
#pragma unroll
    for (int k = 0; k < 8; ++k) row[lane * 8 + k] = 0;
  }
  if (lane == 0) {
    ss.prefix |= (uint64_t)d << dsh;
    ss.mask |= (uint64_t)(nb - 1) << dsh;
    ss.rank -= run;
    s.sel[seg] = ss;
  }
}

// Split: candidates below their segment's chosen bucket are victims; the
// bucket's members go to the list for the remaining digits, with the list's
// key range per segment.
__global__ void __launch_bounds__(256) k_split(DevState s, int single, int fallback) {
  s = with_args(s);
  Ctl* c = s.ctl;
  if (c->status != PS_OK || c->mvict == 0) return;
  if (single && !s.sel[0].active) return;
  {
    // the first digit's 16-bit rows are read: clear them for the next select
    const int nrows = c->wide_nrows;
    if (nrows <= kWideRows) {
      uint4* w = reinterpret_cast<uint4*>(s.wide_bins);
      const int64_t n4 = (int64_t)nrows * kWideBins / 4;
      for (int64_t k = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; k < n4; k += (int64_t)gridDim.x * blockDim.x)
        w[k] = make_uint4(0, 0, 0, 0);
    }
  }
  // the segments' state, once per CTA (s_act: 1 selecting, 2 taken whole)
  __shared__ uint64_t s_pre[PS_MAX_GROUPS], s_msk[PS_MAX_GROUPS];
  __shared__ uint8_t s_act[PS_MAX_GROUPS];
  const int nseg = single ? 1 : s.G;
  const bool whole = !single && s.policy == PS_PREFIXSHIELD;
  for (int g = threadIdx.x; g < nseg; g += blockDim.x) {
    const SelSeg ss = s.sel[g];
    s_pre[g] = ss.prefix;
    s_msk[g] = ss.mask;
    s_act[g] = (whole && s.grp_full[g]) ? 2 : (ss.active ? 1 : 0);
  }
  __syncthreads();
  int marked = 0;
  for (int64_t b0 = blockIdx.x * (int64_t)blockDim.x; b0 < s.N; b0 += (int64_t)gridDim.x * blockDim.x) {
    const int64_t b = b0 + threadIdx.x;
    bool v = false, to_list = false;
    uint64_t key = ~0ull;
    int seg = 0;
    if (b < s.N) {
      key = s.csk[b];
      const int grp = single ? 0 : s.blk_group[b];
      if (key != ~0ull && !(fallback && ((s.bm_victim[b >> 5] >> (b & 31)) & 1))) {
        seg = grp;
        if (s_act[seg] == 2) {
          v = true;
        } else if (s_act[seg]) {
          const uint64_t k = key & s_msk[seg];
          v = k < s_pre[seg];
          to_list = k == s_pre[seg];
        }
      }
    }
    const unsigned bits = __ballot_sync(kFull, v);
    if (bits && lane_id() == 0) atomicOr(s.bm_victim + ((b - lane_id()) >> 5), bits);
    marked += __popc(bits);
    const unsigned lm = __ballot_sync(kFull, to_list);
    if (lm) {
      unsigned long long base = 0;
      if (lane_id() == 0) base = atomicAdd(reinterpret_cast<unsigned long long*>(&c->lst_n), (unsigned long long)__popc(lm));
      base = __shfl_sync(kFull, base, 0);
      if (to_list) {
        const int64_t slot = (int64_t)base + __popc(lm & ((1u << lane_id()) - 1));
        s.lst_key[slot] = key;
        s.lst_blk[slot] = (uint32_t)b;
        s.lst_seg[slot] = (uint16_t)seg;
      }
      // the list's key range per segment (lanes of one segment combined)
      const unsigned peers = __match_any_sync(kFull, to_list ? (uint32_t)seg : ~0u);
      if (to_list) {
        const uint32_t hi = (uint32_t)(key >> 32), lo = (uint32_t)key;
        const uint32_t hmin = __reduce_min_sync(peers, hi), hmax = __reduce_max_sync(peers, hi);
        const uint32_t lmin = __reduce_min_sync(peers, hi == hmin ? lo : ~0u);
        const uint32_t lmax = __reduce_max_sync(peers, hi == hmax ? lo : 0u);
        if (lane_id() == __ffs(peers) - 1) {
          atomicMin(reinterpret_cast<unsigned long long*>(&s.sel[seg].qmin), ((unsigned long long)hmin << 32) | lmin);
          atomicMax(reinterpret_cast<unsigned long long*>(&s.sel[seg].qmax), ((unsigned long long)hmax << 32) | lmax);
        }
      }
    }
  }
  if (lane_id() == 0 && marked) atomic_add_i64(&c->n_victims_marked, marked);
}

// The rest of a select on one CTA, with every segment's state in shared
// memory.  A split list of at most kFinCap members is staged in shared memory
// too; a longer one (rare: a boundary bucket of the first digit holding many
// candidates) is read from global memory in each round.  The segments'
// thresholds come from ranking by counting (lists of at most kFinCountCap
// members) or from the remaining radix digits, one round per digit; then
// Eq. 7's tie rule, then the list's victims.  One launch for every list
// length keeps the step graph free of conditional nodes here.
struct FinSeg {
  uint64_t prefix, mask;
  int64_t rank;
  int32_t active, incl;
};
constexpr size_t kFinSmem = (size_t)kFinCap * 8 + (size_t)kFinCap * 2 + (size_t)kFinRows * kRadixBins * 4 +
                            (size_t)PS_MAX_GROUPS * sizeof(FinSeg);

__global__ void __launch_bounds__(1024) k_list_finish(DevState s, int single) {
  s = with_args(s);
  extern __shared__ __align__(16) unsigned char fin_smem[];
  FinSeg* sl = reinterpret_cast<FinSeg*>(fin_smem);
  uint64_t* lkey = reinterpret_cast<uint64_t*>(sl + PS_MAX_GROUPS);
  uint32_t* fh = reinterpret_cast<uint32_t*>(lkey + kFinCap);
  uint16_t* lseg = reinterpret_cast<uint16_t*>(fh + kFinRows * kRadixBins);
  __shared__ int16_t row_of[PS_MAX_GROUPS];
  __shared__ int16_t seg_of_row[PS_MAX_GROUPS];
  __shared__ int s_nrows;
  Ctl* c = s.ctl;
  if (c->status != PS_OK || c->mvict == 0) return;
  // the debt phase's launch also starts the fallback's select (the groups'
  // final take counts are known here)
  const bool start_fb = !single && s.policy == PS_PREFIXSHIELD;
  if (single && !s.sel[0].active) return;
  const int nseg = single ? 1 : s.G;
  const int64_t n = c->lst_n;
  const bool small = n <= kFinCap;
  const int warp = threadIdx.x >> 5, lane = lane_id();
  for (int g = threadIdx.x; g < nseg; g += blockDim.x) {
    const SelSeg v = list_view(s.sel[g]);
    sl[g] = FinSeg{v.prefix, v.mask, v.rank, v.active, v.incl};
  }
  if (small)
    for (int64_t e = threadIdx.x; e < n; e += blockDim.x) { lkey[e] = s.lst_key[e]; lseg[e] = s.lst_seg[e]; }
  __syncthreads();
  auto key_at = [&](int64_t e) -> uint64_t { return small ? lkey[e] : ldcg_u64(s.lst_key + e); };
  auto seg_at = [&](int64_t e) -> int { return small ? (int)lseg[e] : (int)s.lst_seg[e]; };
  // A short list (the usual case): a segment's threshold key is its member
  // whose rank among the segment's list members (keys are unique) is its
  // remaining rank - 1; each thread ranks one member by counting, so no
  // digit rounds (and their barriers) are needed.
  const bool by_count = small && n <= kFinCountCap;
  if (by_count) {
    for (int e = threadIdx.x; e < n; e += blockDim.x) {
      const int g = lseg[e];
      if (!sl[g].active) continue;
      const uint64_t key = lkey[e];
      int64_t below = 0;
      for (int j = 0; j < n; ++j) below += (lseg[j] == g && lkey[j] < key) ? 1 : 0;
      // one member per segment matches, and the loop reads only the
      // segment's activity and rank, which nothing here writes
      if (below == sl[g].rank - 1) {
        sl[g].prefix = key;
        sl[g].mask = ~0ull;
      }
    }
    __syncthreads();
  }
  for (int iter = 0; !by_count && iter < 8; ++iter) {  // at most 8 digits in a 64-bit key
    {
      int k = 0;
      for (int base = 0; base < nseg; base += blockDim.x) {
        const int g = base + threadIdx.x;
        const bool counts = g < nseg && sl[g].active && next_shift(sl[g].mask) >= 0;
        int tot;
        const int ex = block_excl_scan((int)counts, &tot);
        if (g < nseg) row_of[g] = counts ? (int16_t)(k + ex) : (int16_t)-1;
        if (counts) seg_of_row[k + ex] = (int16_t)g;
        k += tot;
      }
      if (threadIdx.x == 0) s_nrows = k;
      __syncthreads();
    }
    const int nrows = s_nrows;
    if (nrows == 0) break;
    for (int r0 = 0; r0 < nrows; r0 += kFinRows) {
      const int rn = tmin(kFinRows, nrows - r0);
      for (int k = threadIdx.x; k < rn * kRadixBins; k += blockDim.x) fh[k] = 0;
      __syncthreads();
      for (int64_t e0 = 0; e0 < n; e0 += blockDim.x) {
        const int64_t e = e0 + threadIdx.x;
        bool act = false;
        uint32_t idx = 0;
        if (e < n) {
          const int seg = seg_at(e);
          const int row = row_of[seg];
          if (row >= r0 && row < r0 + rn) {
            const uint64_t key = key_at(e);
            if ((key & sl[seg].mask) == sl[seg].prefix) {
              act = true;
              const int sh = next_shift(sl[seg].mask);
              idx = (uint32_t)(row - r0) * kRadixBins + (uint32_t)((key >> sh) & (kRadixBins - 1));
            }
          }
        }
        agg_inc(fh, idx, act);
      }
      __syncthreads();
      for (int r = warp; r < rn; r += blockDim.x >> 5) {
        const int seg = seg_of_row[r0 + r];
        const int sh = next_shift(sl[seg].mask);
        const int64_t rank = sl[seg].rank;
        uint32_t v[kRadixBins / 32];
        uint32_t sum = 0;
#pragma unroll
        for (int j = 0; j < kRadixBins / 32; ++j) { v[j] = fh[r * kRadixBins + lane * (kRadixBins / 32) + j]; sum += v[j]; }
        const uint32_t incl = warp_incl_scan(sum);
        const uint32_t excl = incl - sum;
        if ((uint64_t)excl < (uint64_t)rank && (uint64_t)rank <= (uint64_t)incl) {
          uint32_t run = excl;
          int d = 0;
          for (int j = 0; j < kRadixBins / 32; ++j) {
            if ((uint64_t)rank <= (uint64_t)(run + v[j])) { d = lane * (kRadixBins / 32) + j; break; }
            run += v[j];
          }
          sl[seg].prefix |= (uint64_t)d << sh;
          sl[seg].mask |= (uint64_t)(kRadixBins - 1) << sh;
          sl[seg].rank = rank - run;
        }
      }
      __syncthreads();
    }
  }
  // Eq. 7's tie rule at tau: among the groups holding an item at exactly tau,
  // the sel_k with the smallest candidate keys take it
  if (!single && c->sel_ntie > 0) {
    const int64_t k = c->sel_k;
    for (int g = threadIdx.x; g < nseg; g += blockDim.x) {
      if (!(sl[g].active && sl[g].incl == 2)) continue;
      int rank = 0;
      for (int h = 0; h < nseg; ++h) rank += sl[h].active && sl[h].incl == 2 && sl[h].prefix < sl[g].prefix;
      const bool chosen = rank < k;
      s.grp_x[g] -= chosen ? 0 : 1;
      fh[g] = chosen ? 1 : 0;  // applied after every thread has read the flags
    }
    __syncthreads();
    for (int g = threadIdx.x; g < nseg; g += blockDim.x)
      if (sl[g].active && sl[g].incl == 2) sl[g].incl = (int32_t)fh[g];
    __syncthreads();
  }
  // the list's victims: keys below (or at, if incl) the threshold
  for (int64_t e = threadIdx.x; e < n; e += blockDim.x) {
    const uint64_t key = key_at(e);
    const FinSeg& f = sl[seg_at(e)];
    if (f.active && (key < f.prefix || (f.incl && key == f.prefix))) {
      const uint32_t b = s.lst_blk[e];
      atomicOr(s.bm_victim + (b >> 5), 1u << (b & 31));
    }
  }
  if (start_fb) {
    __syncthreads();  // every reader of segment 0's state is done
    if ((threadIdx.x >> 5) == 0) start_global_select(s, c, 1);
  }
}

// TakeTrueFree (Alg. 2) and the step's id lists (allocated, evicted,
// invalidated), all ascending, from the bitmaps.  Each CTA owns kBmChunk
// bitmap words.  Pass 1 counts each chunk's free, evicted and invalidated
// ids.  Pass 2: the ftake smallest free ids are taken greedily from low ids,
// so a chunk takes min(ftake, free before it + its own) - min(ftake, free
// before it) of its free ids, its lowest ones; with the victims they form the
// allocated set, whose ids become resident.
__device__ __forceinline__ uint32_t free_word(const DevState& s, int64_t w) {
  uint32_t f = ~s.res_bits[w];
  const int64_t hi = (w + 1) * 32;
  if (hi > s.N) f &= (1u << (uint32_t)(32 - (hi - s.N))) - 1u;
  return f;
}
__global__ void __launch_bounds__(kBmChunk) k_bm_count(DevState s) {
  s = with_args(s);
  const Ctl* c = s.ctl;
  if (c->status != PS_OK) return;
  const int64_t w = (int64_t)blockIdx.x * kBmChunk + threadIdx.x;
  const int nchunks = gridDim.x;
  const bool in = w < s.nwords;
  const int nv = in ? __popc(s.bm_victim[w]) : 0;
  const int ni = in ? __popc(s.bm_inval[w]) : 0;
  const int nf = (in && c->ftake > 0) ? __popc(free_word(s, w)) : 0;
  const int tv = block_sum(nv), ti = block_sum(ni), tf = block_sum(nf);
  if (threadIdx.x == 0) {
    s.bm_chunk_cnt[0 * nchunks + blockIdx.x] = tf;
    s.bm_chunk_cnt[1 * nchunks + blockIdx.x] = tv;
    s.bm_chunk_cnt[2 * nchunks + blockIdx.x] = ti;
  }
}
// Counts are packed into one 64-bit word (three 21-bit fields: a chunk holds
// at most 8192 ids of each kind), so one block scan carries all three.
__device__ __forceinline__ uint64_t pack3(uint64_t a, uint64_t b, uint64_t c) { return a | b << 21 | c << 42; }
__device__ __forceinline__ int64_t field3(uint64_t v, int k) { return (int64_t)((v >> (21 * k)) & 0x1FFFFF); }
__global__ void __launch_bounds__(kBmChunk) k_bm_write(DevState s) {
  s = with_args(s);
  Ctl* c = s.ctl;
  if (c->status != PS_OK) return;
  const int64_t w = (int64_t)blockIdx.x * kBmChunk + threadIdx.x;
  const int nchunks = gridDim.x;
  const bool in = w < s.nwords;
  const int64_t ftake = c->ftake;
  // earlier chunks' free, evicted and invalidated ids (summed field by field)
  int64_t fb = 0, vb = 0, ib = 0;
  for (int j = threadIdx.x; j < (int)blockIdx.x; j += blockDim.x) {
    fb += s.bm_chunk_cnt[0 * nchunks + j];
    vb += s.bm_chunk_cnt[1 * nchunks + j];
    ib += s.bm_chunk_cnt[2 * nchunks + j];
  }
  {
    __shared__ int64_t s_before[3][kBmChunk / 32];
    fb = warp_sum(fb); vb = warp_sum(vb); ib = warp_sum(ib);
    if (lane_id() == 0) { s_before[0][threadIdx.x >> 5] = fb; s_before[1][threadIdx.x >> 5] = vb; s_before[2][threadIdx.x >> 5] = ib; }
    __syncthreads();
    fb = vb = ib = 0;
#pragma unroll
    for (int q = 0; q < kBmChunk / 32; ++q) { fb += s_before[0][q]; vb += s_before[1][q]; ib += s_before[2][q]; }
  }
  const int64_t take_here = tmin(ftake, fb + s.bm_chunk_cnt[blockIdx.x]) - tmin(ftake, fb);
  // this word's taken free ids: the chunk's lowest take_here free ids
  const uint32_t f = (in && take_here > 0) ? free_word(s, w) : 0u;
  const uint32_t vic = in ? s.bm_victim[w] : 0u, inv = in ? s.bm_inval[w] : 0u;
  uint64_t tot1;
  const uint64_t ex1 = block_excl_scan<uint64_t>(pack3(__popc(f), __popc(vic), __popc(inv)), &tot1);
  const int64_t fl = field3(ex1, 0);
  const int64_t want = tmin<int64_t>(tmax<int64_t>(take_here - fl, 0), __popc(f));
  // the lowest 'want' set bits of f: everything below the want-th set bit, and it
  const uint32_t taken = want == 0 ? 0u : (want >= 32 ? f : (f & ((2u << __fns(f, 0, (int)want)) - 1u)));
  const uint32_t alloc = taken | vic;
  if (in) s.res_bits[w] |= alloc;  // every allocated id is resident after the step
  uint64_t tot2;
  const uint64_t ex2 = block_excl_scan<uint64_t>((uint64_t)__popc(alloc), &tot2);
  const uint32_t bitsk[3] = {alloc, vic, inv};
  const int64_t basek[3] = {vb + tmin(ftake, fb) + (int64_t)ex2, vb + field3(ex1, 1), ib + field3(ex1, 2)};
  int32_t* outs[3] = {s.out.admitted_ids, s.out.evicted_ids, s.out.invalidated_ids};
#pragma unroll
  for (int k = 0; k < 3; ++k) {
    int64_t o = basek[k];
    for (uint32_t b = bitsk[k]; b; b &= b - 1) {
      if (o < s.max_blocks) outs[k][o] = (int32_t)(w * 32 + __ffs(b) - 1);
      ++o;
    }
  }
  if (blockIdx.x == nchunks - 1 && threadIdx.x == 0) {
    c->n_alloc = vb + tmin(ftake, fb) + (int64_t)tot2;
    c->n_evicted = vb + field3(tot1, 1);
  }
  if (in) {
    s.bm_victim[w] = 0;
    s.bm_inval[w] = 0;
  }
}

// Stage 6: place granted claims (thread per position).  The allocated ids
// (ascending) go to the granted keys in (request, position) order; each new
// block carries the metadata OnCacheFullBlocks attached plus any in-step
// touches.  An allocated id that is still resident is a victim (every victim
// is allocated again in its step): its old content leaves the pool first, in
// the same thread (Alg. 2 Evict: table entry and record), so no other thread
// ever sees the block between its two contents.  Each claim's owning position
// then clears its claim-map slot (no other thread reads it here), and each
// request's first position commits its OnRequest / RecordSuccessfulAdmission
// history update.
__global__ void __launch_bounds__(kThreads) k_insert(DevState s) {
  s = with_args(s);
  Ctl* c = s.ctl;
  if (c->status != PS_OK) return;
  const int64_t pos = blockIdx.x * (int64_t)blockDim.x + threadIdx.x;
  if (pos == 0) c->hist_live += c->hist_new;
  PosRef r;
  bool placed = false, evicted = false;
  uint32_t g = 0, gold = 0;
  if (pos_ref(s, pos, &r)) {
    const uint32_t i = r.i;
    const int si = s.rq_s[i], a = s.rq_a[i];
    g = (uint32_t)s.in_group[i];
    if (r.m == 0) {  // history commit of request i (it has a full block)
      const uint32_t hs = s.rq_hs[i];
      if (hs != kNone) {
        atomicAdd(&s.hist[hs].refadm, 1u);
        if (a > 0) atomicOr(&s.hist[hs].refadm, 0x80000000u);
      }
    }
    const uint32_t slot = r.m >= si ? s.pos_claim[pos] : kNone;  // an own claim
    if (r.m >= si && r.m < si + a) {
      const int64_t rank = (int64_t)s.rq_cbase[i] + (r.m - si);
      const uint32_t b = rank < c->n_alloc ? (uint32_t)s.out.admitted_ids[rank] : kNone;
      if (b >= (uint64_t)s.N) {
        c->internal_error = 1;  // the allocated set is short: never expected
      } else {
        const ClaimEntry e = s.claims[slot];
        const uint64_t key = s.pos_key[pos];
        // the id's old record, loaded together: a resident id is a victim,
        // whose old content (table entry, record) leaves first
        const uint8_t ofl = s.blk_flags[b];
        const uint32_t oslot = s.blk_slot[b];
        const uint64_t okey = s.blk_key[b];
        const uint16_t ogrp = s.blk_group[b];
        if (ofl & 1) {
          table_delete_known(s, oslot, okey, ogrp);
          gold = ogrp;
          evicted = true;
        }
        s.blk_key[b] = key;
        s.blk_group[b] = (uint16_t)g;
        s.blk_contract[b] = (uint8_t)s.rq_cid[i];
        s.blk_prefix[b] = s.rq_p[i];
        s.blk_klass[b] = e.promo != kNone ? (uint8_t)kReuse : s.rq_knew[i];
        // the latest request that touched it: an in-step toucher's stamp, or
        // the owner's own
        const uint64_t st = tmax<uint64_t>(e.stamp, make_stamp(c->stamp_base, s.rq_pbase[i], s.rq_n[i], r.m));
        s.blk_stamp[b] = st;
        if (s.lg_on) s.lg_slot[st - c->stamp_base] = b;
        s.blk_acc[b] = e.tcnt;
        s.blk_freq[b] = e.tcnt;
        s.blk_flags[b] = 1;
        s.blk_slot[b] = table_insert(s, key, g, b);
        placed = true;  // its resident bit was set with the allocated set
      }
    }
    if (slot != kNone) s.claims[slot] = empty_claim();
  }
  agg_stat(s, gold, PS_STAT_EVICTED_BLOCKS, 1, evicted);
  agg_stat(s, gold, PS_STAT_RESIDENT_BLOCKS, -1, evicted);
  agg_stat(s, g, PS_STAT_RESIDENT_BLOCKS, 1, placed);
  const int k = __popc(__ballot_sync(kFull, placed)) - __popc(__ballot_sync(kFull, evicted));
  if (lane_id() == 0 && k) atomic_add_i64(&c->n_resident, k);
}

// Step end: the outputs' counts and status, then the clock, the step index
// and the next step's first recency stamp.
__global__ void k_finalize(DevState s) {
  s = with_args(s);
  Ctl* c = s.ctl;
  if (threadIdx.x != 0 || blockIdx.x != 0) return;
  const int32_t st = c->internal_error ? PS_ERR_DEVICE_STATUS : c->status;
  s.out.counts[3] = st;
  if (c->status != PS_OK) return;
  s.out.counts[0] = (int32_t)c->need;
  s.out.counts[1] = (int32_t)c->n_evicted;
  s.out.counts[2] = (int32_t)c->n_inval;
  c->t_prev = s.now;
  c->step += 1;
  c->stamp_base += c->nblocks;
  if (s.policy == PS_S3FIFO) {  // the queue arrays the step wrote become current
    const S3Plan* pl = s.s3_plan;
    const int64_t n_ins = c->need < c->n_alloc ? c->need : c->n_alloc;
    c->s3_len[0] = pl->nKeepS + n_ins - pl->hits;
    c->s3_len[1] = pl->nKeepM + pl->nMid + pl->hits;
    c->s3_buf ^= 1;
    c->s3_ctr = pl->ctr_end + (uint64_t)n_ins;
    c->ghost_live -= pl->hits;
    c->s3_nS = c->s3_len[0];
    c->s3_nM = c->s3_len[1];
  }
}

// Read-only probe output: h_i per request, and the probe's status.
__global__ void k_probe_out(DevState s, int32_t* out, int32_t* status) {
  s = with_args(s);
  const Ctl* c = s.ctl;
  const int i = blockIdx.x * blockDim.x + threadIdx.x;
  if (i == 0) *status = c->status;
  if (c->status != PS_OK || i >= s.R) return;
  out[i] = s.rq_h[i];
}

// ===========================================================================
// host launchers
static int grid_for(int64_t items, int threads, int max_ctas) {
  int64_t g = (items + threads - 1) / threads;
  if (g < 1) g = 1;
  if (g > max_ctas) g = max_ctas;
  return (int)g;
}

void launch_init(const DevState& s, cudaStream_t st) {
  k_init_blocks<<<grid_for((int64_t)kClaimWays << s.cl_nbuckets_log2, 256, 152 * 8), 256, 0, st>>>(s);
  k_init_ctl<<<1, 1024, 0, st>>>(s);
  launch_queue_init(s, st);
}

template <int BS>
static void launch_hash_lookup_t(const DevState& s, cudaStream_t st, int probe) {
  // persistent: the CTAs that fit at once (more only queue behind them)
  int dev = 0, nsm = 152;
  if (cudaGetDevice(&dev) == cudaSuccess) cudaDeviceGetAttribute(&nsm, cudaDevAttrMultiProcessorCount, dev);
  const int64_t want = (s.max_segments + 7) / 8;
  const int grid = (int)(want < (int64_t)nsm * kHashCtasPerSm ? want : (int64_t)nsm * kHashCtasPerSm);
  k_hash_lookup<BS><<<grid > 0 ? grid : 1, 256, 0, st>>>(s, probe);
}
static int32_t launch_hash_lookup(const DevState& s, cudaStream_t st, int probe) {
  switch (s.bs) {
    case 2: launch_hash_lookup_t<2>(s, st, probe); break;
    case 4: launch_hash_lookup_t<4>(s, st, probe); break;
    case 8: launch_hash_lookup_t<8>(s, st, probe); break;
    case 16: launch_hash_lookup_t<16>(s, st, probe); break;
    case 32: launch_hash_lookup_t<32>(s, st, probe); break;
    case 64: launch_hash_lookup_t<64>(s, st, probe); break;
    default: return PS_ERR_INVALID_ARG;
  }
  return PS_OK;
}

void configure_kernels(const DevState& s) {
  (void)s;
  cudaFuncSetAttribute(k_list_finish, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kFinSmem);
  cudaFuncSetAttribute(k_cand, cudaFuncAttributeMaxDynamicSharedMemorySize, PS_MAX_GROUPS * kClasses * 5 * 4);
  cudaFuncSetAttribute(k_grant, cudaFuncAttributeMaxDynamicSharedMemorySize, PS_MAX_GROUPS * PS_MAX_CONTRACTS * 8);
}

int32_t launch_step(const DevState& s, cudaStream_t st, StepTrace* tr, const CaptureCtx* cap) {
  // grids depend only on the handle's bounds (a captured graph serves any step)
  const int R = s.max_requests;
  const int pgrid = grid_for(s.max_blocks, kThreads, 1 << 30);
  const int prgrid = grid_for(s.max_blocks + R, kThreads, 1 << 30);
  const int ngrid = grid_for(s.N, 256, 152 * 8);
  const int sgrid = grid_for(s.N, 256, 152 * 4);  // 48 KB histograms: 4 CTAs per SM
  const int cgrid = grid_for(s.N, 256, 152 * 8);
  int launches = 0;
  auto mark = [&](int stage) {
    // under capture an external record becomes an event-record node of the
    // graph (the flag is refused outside a capture)
    if (tr && tr->timing) {
      if (cap) cudaEventRecordWithFlags(tr->ev[stage], st, cudaEventRecordExternal);
      else cudaEventRecord(tr->ev[stage], st);
    }
  };
#define PS_LAUNCH(...) do { __VA_ARGS__; ++launches; } while (0)
  mark(0);
  PS_LAUNCH(launch_k(k_validate, grid_for(R, kValTile, 1 << 20), kValTile, 0, st, s, 0));
  mark(1);
  if (launch_hash_lookup(s, st, 0) != PS_OK) return PS_ERR_INVALID_ARG;
  ++launches;
  mark(2);
  PS_LAUNCH(launch_k(k_claims, prgrid, kThreads, 0, st, s));
  mark(3);
  // The candidates read pins and residency (final from here on) and the class
  // and stamp of unpinned blocks, which S3-S4 leave alone: under capture
  // they are counted on a side branch that runs beside the rest of S3-S4.
  // The candidate scan writes per-step scratch only, so it forks before the
  // grants (a step the grant then fails ignores what it wrote); the indexed
  // queues' count applies the step's pins to persistent counts, so it waits
  // for the grant's verdict.
  const bool fork = cap && s.policy != PS_S3FIFO;
  const bool early = fork && !s.lg_on;
  cudaStream_t cs = st;
  auto launch_cand = [&]() -> int32_t {
    if (fork) {
      if (cudaEventRecord(cap->fork, st) != cudaSuccess || cudaStreamWaitEvent(cap->side, cap->fork, 0) != cudaSuccess)
        return PS_ERR_CUDA;
      cs = cap->side;
    }
    const int cand_smem = (s.policy == PS_PREFIXSHIELD || s.policy == PS_STATICQUOTA ? s.G : 1) * kClasses * 5 * 4;
    if (s.lg_on) {
      if (launch_queue_cand(s, cs, &launches) != PS_OK) return PS_ERR_CUDA;
    } else if (s.policy != PS_S3FIFO) {
      // one 512-thread CTA per SM: the main branch keeps room on every SM
      PS_LAUNCH(k_cand<<<fork ? 152 : grid_for(s.N, 1024 * 4, 152), fork ? 512 : 1024, cand_smem, cs>>>(s));
    }
    if (fork && cudaEventRecord(cap->join, cs) != cudaSuccess) return PS_ERR_CUDA;
    return PS_OK;
  };
  if (early && launch_cand() != PS_OK) return PS_ERR_CUDA;
  if (s.policy == PS_STATICQUOTA) PS_LAUNCH(launch_k(k_grant_quota, s.G, 1024, 0, st, s));
  PS_LAUNCH(launch_k(k_grant, 1, 1024, (size_t)s.G * s.C * 8, st, s));
  if (!early && launch_cand() != PS_OK) return PS_ERR_CUDA;
  // The in-step hits, the metering and the touch passes feed the insertion
  // (the claims' in-step touches, the new blocks' class) and the statistics;
  // the select needs only the step's debts, which k_grant settles.  Under
  // capture they run on a second parallel branch beside the select, joined
  // before the insertion (which reads, then clears, the claim entries).
  // The S3-FIFO select reads only unpinned blocks' frequencies, pin tags and
  // residency, none of which these kernels write (a touch changes hit, so
  // pinned, blocks), so it runs beside them too.  The indexed queues keep
  // them in line (their select reads the touched blocks' new stamps).
  const bool fork2 = cap != nullptr && !s.lg_on;
  cudaStream_t ms = st;
  if (fork2) {
    if (cudaEventRecord(cap->fork2, st) != cudaSuccess || cudaStreamWaitEvent(cap->side2, cap->fork2, 0) != cudaSuccess)
      return PS_ERR_CUDA;
    ms = cap->side2;
  }
  PS_LAUNCH(launch_k(k_instep, pgrid, kThreads, 0, ms, s));
  mark(4);
  PS_LAUNCH(launch_k(k_meter, s.G, 512, 0, ms, s));
  mark(5);
  PS_LAUNCH(launch_k(k_touch, pgrid, kThreads, 0, ms, s));
  PS_LAUNCH(launch_k(k_touch2, pgrid, kThreads, 0, ms, s));
  if (fork2 && cudaEventRecord(cap->join2, cap->side2) != cudaSuccess) return PS_ERR_CUDA;
  mark(6);
  if (fork && cudaStreamWaitEvent(st, cap->join, 0) != cudaSuccess) return PS_ERR_CUDA;
  if (s.lg_on) {
    // indexed queues: the same victims, taken from the queues' heads
    cudaGraphConditionalHandle hq_fb = 0;
    if (s.policy == PS_PREFIXSHIELD) {
      if (cap && !cond_handle(st, &hq_fb)) return PS_ERR_CUDA;
      // the first kernel after the side branch's join depends on two nodes:
      // a plain launch (a programmatic edge takes a single kernel predecessor)
      PS_LAUNCH(k_waterfill<<<1, 1024, 0, st>>>(s, hq_fb, cap ? 1 : 0));
      if (launch_queue_select(s, st, cap, 0, 0, false, &launches) != PS_OK) return PS_ERR_CUDA;
      cudaStream_t f = st;
      if (cap) {
        if (!cond_open(st, cap->aux, hq_fb)) return PS_ERR_CUDA;
        f = cap->aux;
      }
      if (launch_queue_select(s, f, cap, 1, 1, false, &launches) != PS_OK) return PS_ERR_CUDA;
      if (cap && !cond_close(cap->aux)) return PS_ERR_CUDA;
    } else if (launch_queue_select(s, st, cap, s.policy == PS_LRU ? 2 : 3, 0, fork, &launches) != PS_OK) {
      return PS_ERR_CUDA;
    }
  }
  // One exact segmented select: a digit over the candidates, the split, then
  // the split list finished by one CTA.  Every phase is launched on every
  // step (a kernel of a phase with nothing to select returns at once): a
  // conditional graph node measured about 10 us a step even when its body
  // was skipped, more than the phase's early-returning launches.
  auto select = [&](int single, int fallback) {
    PS_LAUNCH(launch_k(k_wide_pass, cgrid, 256, 0, st, s, single, fallback));
    PS_LAUNCH(launch_k(k_wide_resolve, single ? 1 : s.G, 32, 0, st, s, single));
    PS_LAUNCH(launch_k(k_split, cgrid, 256, 0, st, s, single, fallback));
    PS_LAUNCH(launch_k(k_list_finish, 1, 1024, kFinSmem, st, s, single));
  };
  if (s.lg_on) {
    // selected above
  } else if (s.policy == PS_PREFIXSHIELD) {
    PS_LAUNCH(k_waterfill<<<1, 1024, 0, st>>>(s, 0, 0));  // after the join: plain
    select(0, 0);
    select(1, 1);  // the global fallback, started by the debt phase's finish
  } else if (s.policy == PS_STATICQUOTA) {
    PS_LAUNCH(k_quota_sel<<<1, 1024, 0, st>>>(s));  // after the join: plain
    select(0, 0);
  } else if (s.policy == PS_LRU) {
    PS_LAUNCH(k_sel_single<<<1, 32, 0, st>>>(s, 0));  // after the join: plain
    select(1, 0);
  } else if (launch_s3_select(s, st, fork2, &launches) != PS_OK) {
    return PS_ERR_CUDA;
  }
  mark(7);
  const int nchunks = (int)((s.nwords + kBmChunk - 1) / kBmChunk);
  PS_LAUNCH(launch_k(k_bm_count, nchunks, kBmChunk, 0, st, s));
  PS_LAUNCH(launch_k(k_bm_write, nchunks, kBmChunk, 0, st, s));
  mark(8);
  // (evictions happen in k_insert: every victim is allocated again in its step)
  mark(9);
  if (fork2) {  // the touch branch joins the insertion
    if (cudaStreamWaitEvent(st, cap->join2, 0) != cudaSuccess) return PS_ERR_CUDA;
    PS_LAUNCH((k_insert<<<pgrid, kThreads, 0, st>>>(s)));  // after the join: plain
  } else {
    PS_LAUNCH(launch_k(k_insert, pgrid, kThreads, 0, st, s));
  }
  if (s.policy == PS_S3FIFO && launch_s3_insert(s, st, &launches) != PS_OK) return PS_ERR_CUDA;
  if (s.lg_on && launch_queue_append(s, st, cap, &launches) != PS_OK) return PS_ERR_CUDA;
  mark(10);
  PS_LAUNCH(launch_k(k_finalize, 1, 32, 0, st, s));
  mark(11);
#undef PS_LAUNCH
  if (tr) tr->launches = launches;
  return cudaGetLastError() == cudaSuccess ? PS_OK : PS_ERR_CUDA;
}

// The step's outputs into the caller's page-locked host buffers (one pass,
// grid-stride; the id lists by the counts the step wrote).
__global__ void __launch_bounds__(256) k_host_out(ps_step_out_t d, ps_step_out_t h, int32_t R, int32_t G) {
  const int64_t t = blockIdx.x * (int64_t)blockDim.x + threadIdx.x, nt = (int64_t)gridDim.x * blockDim.x;
  const bool ok = d.counts[3] == PS_OK;
  const int64_t n0 = ok ? d.counts[0] : 0, n1 = ok ? d.counts[1] : 0, n2 = ok ? d.counts[2] : 0;
  if (h.counts && t < 4) h.counts[t] = d.counts[t];
  for (int64_t i = t; i < R; i += nt) {
    if (h.hit_blocks) h.hit_blocks[i] = d.hit_blocks[i];
    if (h.admitted_blocks) h.admitted_blocks[i] = d.admitted_blocks[i];
  }
  if (h.admitted_offsets)
    for (int64_t i = t; i <= R; i += nt) h.admitted_offsets[i] = d.admitted_offsets[i];
  for (int64_t i = t; i < G; i += nt) {
    if (h.debt_raw) h.debt_raw[i] = d.debt_raw[i];
    if (h.debt_norm) h.debt_norm[i] = d.debt_norm[i];
  }
  if (h.admitted_ids)
    for (int64_t i = t; i < n0; i += nt) h.admitted_ids[i] = d.admitted_ids[i];
  if (h.evicted_ids)
    for (int64_t i = t; i < n1; i += nt) h.evicted_ids[i] = d.evicted_ids[i];
  if (h.invalidated_ids)
    for (int64_t i = t; i < n2; i += nt) h.invalidated_ids[i] = d.invalidated_ids[i];
}

void launch_host_out(const ps_step_out_t& dev, const ps_step_out_t& host, int32_t R, int32_t G, cudaStream_t st) {
  k_host_out<<<152 * 2, 256, 0, st>>>(dev, host, R, G);
}

int32_t launch_probe(const DevState& s, cudaStream_t st, int32_t* out, int32_t* status) {
  const int rgrid = grid_for(s.R, 256, 1 << 20);
  const int pgrid = grid_for(s.max_blocks, kThreads, 1 << 30);
  DevState p = s;
  p.args = nullptr;  // the probe's kernels take every argument by value
  k_validate<<<grid_for(p.max_requests, kValTile, 1 << 20), kValTile, 0, st>>>(p, 1);
  if (s.R > 0 && launch_hash_lookup(p, st, 1) != PS_OK) return PS_ERR_INVALID_ARG;
  k_probe_out<<<rgrid, 256, 0, st>>>(p, out, status);
  return cudaGetLastError() == cudaSuccess ? PS_OK : PS_ERR_CUDA;
}

}  // namespace ps
