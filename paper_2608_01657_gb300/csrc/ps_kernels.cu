// Kernels of the batched prefix-cache step (PrefixShield, arXiv 2608.01657).
//
// One step is a fixed sequence of launches on the caller's stream.  Nothing on
// the path goes back to the host: every size (tokens, blocks, claims, victims)
// lives in device memory, and a kernel whose work is empty exits at once.
// Each kernel's comment names the stage and the passage it implements.
#include <climits>
#include <cstdio>

#include "ps_internal.cuh"

namespace ps {

constexpr unsigned kFull = 0xFFFFFFFFu;
constexpr int kWarpsPerCta = 8;  // warp-per-request kernels

// ---------------------------------------------------------------------------
// small device helpers
__device__ __forceinline__ int lane_id() { return threadIdx.x & 31; }
template <typename T>
__device__ __forceinline__ T tmin(T a, T b) { return a < b ? a : b; }
template <typename T>
__device__ __forceinline__ T tmax(T a, T b) { return a < b ? b : a; }

template <typename T>
__device__ __forceinline__ T warp_incl_scan(T v) {
  const int lane = lane_id();
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    T n = __shfl_up_sync(kFull, v, o);
    if (lane >= o) v += n;
  }
  return v;
}
template <typename T>
__device__ __forceinline__ T warp_sum(T v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(kFull, v, o);
  return v;
}

// Exclusive scan across the CTA (blockDim a multiple of 32).  Returns the
// thread's exclusive prefix and writes the CTA total to *total.
template <typename T>
__device__ T block_excl_scan(T v, T* total) {
  __shared__ T wsum[32];
  const int lane = lane_id(), warp = threadIdx.x >> 5, nw = blockDim.x >> 5;
  T incl = warp_incl_scan(v);
  if (lane == 31) wsum[warp] = incl;
  __syncthreads();
  if (warp == 0) {
    T w = lane < nw ? wsum[lane] : T(0);
    T wi = warp_incl_scan(w);
    __syncwarp();
    wsum[lane] = wi;
  }
  __syncthreads();
  T base = warp ? wsum[warp - 1] : T(0);
  *total = wsum[nw - 1];
  __syncthreads();
  return base + incl - v;
}
template <typename T>
__device__ T block_sum(T v) {
  T tot;
  block_excl_scan(v, &tot);
  return tot;
}

__device__ __forceinline__ void atomic_add_i64(int64_t* p, int64_t v) {
  atomicAdd(reinterpret_cast<unsigned long long*>(p), static_cast<unsigned long long>(v));
}
__device__ __forceinline__ int64_t& stat_ref(const DevState& s, int g, int k) {
  return s.stats[(int64_t)g * PS_NUM_STATS + k];
}
// Warp-aggregated increment of bins[idx] for the lanes with 'active'.
__device__ __forceinline__ void agg_inc(uint32_t* bins, uint32_t idx, bool active) {
  unsigned act = __ballot_sync(kFull, active);
  if (!active) return;
  unsigned peers = __match_any_sync(act, idx);
  if (lane_id() == __ffs(peers) - 1) atomicAdd(bins + idx, (uint32_t)__popc(peers));
}
__device__ __forceinline__ uint64_t ldcg_u64(const uint64_t* p) { return __ldcg(reinterpret_cast<const unsigned long long*>(p)); }
__device__ __forceinline__ uint32_t ldcg_u32(const uint32_t* p) { return __ldcg(p); }

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
  int64_t need = beta - b;
  if (need <= 0 || dt >= (need + rho - 1) / rho) return beta;
  return b + rho * dt;
}
__device__ __forceinline__ int64_t muldiv(int64_t a, int64_t b, int64_t c) {
  return (int64_t)(((__int128)a * (__int128)b) / (__int128)c);
}

// ---- native prefix table ---------------------------------------------------
// Lookup of 4 keys per warp, 8 lanes per key: each lane loads one 16-byte
// entry of the key's 128-byte bucket.  A bucket whose overflow count is zero
// ends the probe.  Returns (for lane m in [kk, kk+4)) the block of key kk+...
__device__ uint32_t table_lookup4(const DevState& s, uint64_t key_of_group, uint32_t g, bool act_in) {
  const int lane = lane_id();
  const uint32_t mask = (1u << s.tb_nbuckets_log2) - 1;
  bool act = act_in;
  uint32_t b = table_home(key_of_group, g, s.tb_nbuckets_log2);
  uint32_t found = kNone;
  for (uint32_t it = 0; it <= mask; ++it) {
    bool hit = false;
    uint32_t eblk = kNone;
    if (act) {
      const uint4 raw = __ldcg(reinterpret_cast<const uint4*>(s.table + (size_t)b * kTableWays + (lane & 7)));
      const uint64_t ek = ((uint64_t)raw.y << 32) | raw.x;
      eblk = raw.z;
      hit = eblk != kNone && ek == key_of_group && raw.w == g;
    }
    const unsigned mh = __ballot_sync(kFull, hit);
    const unsigned gm = (mh >> (lane & ~7)) & 0xFFu;
    const int src = gm ? (lane & ~7) + __ffs(gm) - 1 : lane;
    const uint32_t v = __shfl_sync(kFull, eblk, src);
    if (act) {
      if (gm) {
        found = v;
        act = false;
      } else if (ldcg_u32(s.table_ovf + b) == 0) {
        act = false;
      } else {
        b = (b + 1) & mask;
      }
    }
    if (!__any_sync(kFull, act)) break;
  }
  return found;
}

__device__ uint32_t table_insert(const DevState& s, uint64_t key, uint32_t g, uint32_t blk) {
  const uint32_t mask = (1u << s.tb_nbuckets_log2) - 1;
  uint32_t b = table_home(key, g, s.tb_nbuckets_log2);
  for (uint32_t it = 0; it <= mask; ++it) {
    for (int w = 0; w < kTableWays; ++w) {
      TableEntry* e = s.table + (size_t)b * kTableWays + w;
      if (ldcg_u32(&e->blk) == kNone && atomicCAS(&e->blk, kNone, blk) == kNone) {
        e->key = key;
        e->grp = g;
        return b * kTableWays + w;
      }
    }
    atomicAdd(s.table_ovf + b, 1u);
    b = (b + 1) & mask;
  }
  return kNone;  // unreachable: the table is at most half full
}

__device__ void table_delete(const DevState& s, uint32_t blk) {
  const uint32_t mask = (1u << s.tb_nbuckets_log2) - 1;
  const uint32_t slot = s.blk_slot[blk];
  const uint32_t bucket = slot / kTableWays;
  uint32_t x = table_home(s.blk_key[blk], s.blk_group[blk], s.tb_nbuckets_log2);
  TableEntry* e = s.table + slot;
  e->key = 0;
  e->grp = 0;
  e->blk = kNone;
  for (uint32_t it = 0; x != bucket && it <= mask; ++it, x = (x + 1) & mask) atomicSub(s.table_ovf + x, 1u);
}

// ---- per-step claim map ------------------------------------------------------
__device__ uint32_t claim_insert(const DevState& s, uint64_t key, uint32_t req) {
  const uint32_t mask = (1u << s.cl_nbuckets_log2) - 1;
  uint32_t b = claim_home(key, s.cl_nbuckets_log2);
  for (uint32_t it = 0; it <= mask; ++it) {
    for (int w = 0; w < kClaimWays; ++w) {
      ClaimEntry* e = s.claims + (size_t)b * kClaimWays + w;
      uint64_t cur = ldcg_u64(&e->key);
      if (cur == 0)
        cur = atomicCAS(reinterpret_cast<unsigned long long*>(&e->key), 0ull, (unsigned long long)key);
      if (cur == 0 || cur == key) {
        atomicMin(&e->minreq, req);
        return b * kClaimWays + w;
      }
    }
    b = (b + 1) & mask;
  }
  return kNone;  // unreachable: the map is sized for twice the blocks of a step
}

// ---- block state changes -----------------------------------------------------
// Remove a resident block from the pool (eviction or invalidation).
__device__ void drop_block(const DevState& s, uint32_t b, int stat_kind) {
  table_delete(s, b);
  const int g = s.blk_group[b];
  const uint8_t fl = s.blk_flags[b];
  s.blk_flags[b] = 0;
  atomicAnd(s.res_bits + (b >> 5), ~(1u << (b & 31)));
  atomic_add_i64(&s.ctl->n_resident, -1);
  atomic_add_i64(&stat_ref(s, g, stat_kind), 1);
  atomic_add_i64(&stat_ref(s, g, PS_STAT_RESIDENT_BLOCKS), -1);
  if (s.policy == PS_S3FIFO) atomic_add_i64((fl & 2) ? &s.ctl->s3_nM : &s.ctl->s3_nS, -1);
}

// ===========================================================================
// Init: an empty pool, every balance at beta (Sec. III-B, B = beta at t = 0).
__global__ void k_init_blocks(DevState s) {
  for (int64_t b = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; b < s.N; b += (int64_t)gridDim.x * blockDim.x) {
    s.blk_flags[b] = 0;
    s.blk_pin[b] = 0;
    s.blk_inval[b] = 0;
    s.blk_promo[b] = 0;
  }
  const int64_t nclaims = (int64_t)kClaimWays << s.cl_nbuckets_log2;
  for (int64_t c = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; c < nclaims; c += (int64_t)gridDim.x * blockDim.x) {
    ClaimEntry e{};
    e.key = 0; e.minreq = kNone; e.last = 0; e.tcnt = 0; e.promo = kNone; e.pad0 = 0; e.pad1 = 0;
    s.claims[c] = e;
  }
}
__global__ void k_init_ctl(DevState s) {
  if (threadIdx.x == 0 && blockIdx.x == 0) {
    Ctl c{};
    c.step = 1;
    *s.ctl = c;
  }
  for (int i = threadIdx.x; i < s.G * s.C; i += blockDim.x) s.ledger[i] = s.beta[i % s.C];
}

// ===========================================================================
// Stage 0: validation of the step's inputs; n_i and block positions.
__global__ void __launch_bounds__(1024) k_validate(DevState s) {
  Ctl* c = s.ctl;
  __shared__ int s_bad;
  if (threadIdx.x == 0) s_bad = 0;
  __syncthreads();
  const int R = s.R;
  for (int i = threadIdx.x; i < R; i += blockDim.x) {
    const int64_t o0 = s.in_offsets[i], o1 = s.in_offsets[i + 1];
    const int g = s.in_group[i];
    bool bad = o1 < o0 || g < 0 || g >= s.G || (o1 - o0) / s.bs > (int64_t)kMaxPos;
    if (s.in_contract) bad |= s.in_contract[i] < 0 || s.in_contract[i] >= s.C;
    if (s.in_prefix) bad |= s.in_prefix[i] == 0;
    if (bad) atomicOr(&s_bad, 1);
  }
  __syncthreads();
  int32_t st = PS_OK;
  const int64_t T = R > 0 ? s.in_offsets[R] : 0;
  if (c->sticky != PS_OK) st = c->sticky;
  else if (s.now < c->t_prev) st = PS_ERR_CLOCK;
  else if (c->step > kMaxStep) st = PS_ERR_CAPACITY;
  else if (s_bad || (R > 0 && s.in_offsets[0] != 0) || T > s.max_tokens) st = PS_ERR_INVALID_ARG;
  if (st != PS_OK) {
    if (threadIdx.x == 0) c->status = st;
    return;
  }
  int32_t carry = 0;
  for (int t0 = 0; t0 < R; t0 += blockDim.x) {
    const int i = t0 + threadIdx.x;
    int32_t n = 0;
    if (i < R) {
      n = (int32_t)((s.in_offsets[i + 1] - s.in_offsets[i]) / s.bs);
      s.rq_n[i] = n;
      s.rq_cid[i] = s.in_contract ? s.in_contract[i] : s.contract_of_group[s.in_group[i]];
    }
    int32_t tot;
    const int32_t ex = block_excl_scan(n, &tot);
    if (i < R) s.rq_pbase[i] = carry + ex;
    carry += tot;
  }
  if (threadIdx.x == 0) {
    c->status = PS_OK;
    c->T = T;
    c->nblocks = carry;
    c->pinned = 0; c->n_inval = 0; c->total_claims = 0; c->avail = 0; c->need = 0;
    c->nfree = 0; c->ftake = 0; c->mvict = 0; c->hist_new = 0; c->n_evicted = 0;
    c->n_alloc = 0; c->n_victims_marked = 0; c->m_fb = 0; c->sel_ntie = 0; c->sel_k = 0; c->ticket = 0;
    c->internal_error = 0;
  }
}

// ===========================================================================
// Stages 1-2: chained block hashing and longest cached prefix, one warp per
// request (Sec. III-B native content key; n_cached of Alg. 1).
//
// Tokens of 32 blocks at a time are staged in shared memory with coalesced
// 16-byte loads.  NH products are spread over the warp: lane l takes pair
// (l % PPB) of block (l / PPB + (32 / PPB) r) in round r, PPB = bs / 2; the
// pair sums are reduced with xor shuffles and routed to lane = block.  The
// chain h_m = mix(mix(h_{m-1} ^ NH0) ^ NH2 ^ m) is then serial over the lanes.
// Every key is looked up in the table; the first miss ends the cached prefix
// h_i; blocks before it are pinned; every position at or past it is claimed in
// the step's claim map (lowest request index wins, invariant I1).
template <int PPB>
__global__ void __launch_bounds__(kWarpsPerCta * 32) k_hash_lookup(DevState s) {
  extern __shared__ int32_t smem_tokens[];
  if (s.ctl->status != PS_OK) return;
  constexpr int BS = 2 * PPB;
  constexpr int G32 = 32 / PPB;
  const int warp = threadIdx.x >> 5, lane = lane_id();
  const int i = blockIdx.x * kWarpsPerCta + warp;
  if (i >= s.R) return;
  int32_t* buf = smem_tokens + warp * (32 * BS + 4);
  const uint32_t g = (uint32_t)s.in_group[i];
  const int64_t o0 = s.in_offsets[i];
  const int n = s.rq_n[i];
  const int pbase = s.rq_pbase[i];
  const int64_t T = s.ctl->T;
  const uint32_t step32 = (uint32_t)s.ctl->step;
  const int k = lane % PPB;
  const uint32_t K0 = s.key_words[2 * k], K1 = s.key_words[2 * k + 1];
  const uint32_t K2 = s.key_words[2 * k + 2], K3 = s.key_words[2 * k + 3];
  uint64_t h = chain_seed(s.hash_seed, (int32_t)g);
  uint64_t key0 = 0;
  int hfirst = -1;
  int pinned_new = 0;
  for (int c0 = 0; c0 < n; c0 += 32) {
    const int nb = min(32, n - c0);
    const int64_t cs = o0 + (int64_t)c0 * BS, ce = cs + (int64_t)nb * BS;
    if (s.tokens_aligned16) {
      const int64_t q1 = (ce + 3) >> 2;
      for (int64_t q = (cs >> 2) + lane; q < q1; q += 32) {
        const int64_t t0 = q << 2;
        int v[4];
        if (t0 + 3 < T) {
          const int4 w = __ldcs(reinterpret_cast<const int4*>(s.in_tokens) + q);
          v[0] = w.x; v[1] = w.y; v[2] = w.z; v[3] = w.w;
        } else {
#pragma unroll
          for (int j = 0; j < 4; ++j) v[j] = (t0 + j < T) ? s.in_tokens[t0 + j] : 0;
        }
#pragma unroll
        for (int j = 0; j < 4; ++j)
          if (t0 + j >= cs && t0 + j < ce) buf[t0 + j - cs] = v[j];
      }
    } else {
      for (int64_t t = cs + lane; t < ce; t += 32) buf[t - cs] = s.in_tokens[t];
    }
    __syncwarp();
    uint64_t d1 = 0, d2 = 0;
#pragma unroll
    for (int r = 0; r < PPB; ++r) {
      const int b = lane / PPB + G32 * r;
      uint64_t p1 = 0, p2 = 0;
      if (b < nb) {
        const int2 t = *reinterpret_cast<const int2*>(buf + b * BS + 2 * k);
        p1 = (uint64_t)((uint32_t)t.x + K0) * (uint64_t)((uint32_t)t.y + K1);
        p2 = (uint64_t)((uint32_t)t.x + K2) * (uint64_t)((uint32_t)t.y + K3);
      }
#pragma unroll
      for (int off = 1; off < PPB; off <<= 1) {
        p1 += __shfl_xor_sync(kFull, p1, off);
        p2 += __shfl_xor_sync(kFull, p2, off);
      }
      const int src = (lane % G32) * PPB;
      const uint64_t q1 = __shfl_sync(kFull, p1, src), q2 = __shfl_sync(kFull, p2, src);
      if (lane / G32 == r) { d1 = q1; d2 = q2; }
    }
    __syncwarp();
    uint64_t key = 0;
    for (int j = 0; j < nb; ++j) {
      const uint64_t x = __shfl_sync(kFull, d1, j), y = __shfl_sync(kFull, d2, j);
      h = fix_reserved(mix64(mix64(h ^ x) ^ y ^ (uint64_t)(c0 + j)));
      if (lane == j) key = h;
    }
    if (c0 == 0) key0 = __shfl_sync(kFull, key, 0);
    const bool valid = lane < nb;
    const int pos = pbase + c0 + lane;
    if (valid) s.pos_key[pos] = key;
    // lookup, 4 keys per pass
    uint32_t blk = kNone;
    for (int kk = 0; kk < nb; kk += 4) {
      const int my = kk + (lane >> 3);
      const uint64_t kkey = __shfl_sync(kFull, key, my & 31);
      const uint32_t f = table_lookup4(s, kkey, g, my < nb);
      const uint32_t r = __shfl_sync(kFull, f, ((lane - kk) & 3) * 8);
      if (lane >= kk && lane < kk + 4) blk = r;
    }
    if (valid) s.pos_blk[pos] = blk;
    const unsigned miss = __ballot_sync(kFull, valid && blk == kNone);
    if (hfirst < 0 && miss) hfirst = c0 + __ffs(miss) - 1;
    const int hcur = hfirst < 0 ? INT_MAX : hfirst;
    const int m = c0 + lane;
    bool newpin = false;
    if (valid) {
      if (m < hcur) {
        newpin = atomicExch(s.blk_pin + blk, step32) != step32;
        s.pos_claim[pos] = kNone;
      } else {
        s.pos_claim[pos] = claim_insert(s, key, (uint32_t)i);
      }
    }
    pinned_new += __popc(__ballot_sync(kFull, newpin));
  }
  const int h_i = hfirst < 0 ? n : hfirst;
  if (lane == 0) {
    s.rq_h[i] = h_i;
    if (pinned_new) atomic_add_i64(&s.ctl->pinned, pinned_new);
    uint32_t hs = kNone;
    uint64_t p = 0;
    if (n > 0) {
      p = s.in_prefix ? s.in_prefix[i] : key0;
      const uint32_t hmask = (1u << s.hist_cap_log2) - 1;
      uint32_t x = hist_home(p, g, s.hist_cap_log2);
      for (uint32_t it = 0; it <= hmask; ++it, x = (x + 1) & hmask) {
        uint64_t olo, ohi;
        cas128(s.hist + x, 0ull, 0ull, p, (uint64_t)(g + 1), &olo, &ohi);
        if (olo == 0 && ohi == 0) {
          atomic_add_i64(&s.ctl->hist_new, 1);
          hs = x;
          break;
        }
        if (olo == p && (uint32_t)ohi == g + 1) {
          hs = x;
          break;
        }
      }
      if (hs != kNone)
        atomicMax(reinterpret_cast<unsigned long long*>(&s.hist[hs].ftag),
                  (unsigned long long)step_tag(s.ctl->step, (uint32_t)i));
    }
    s.rq_hs[i] = hs;
    s.rq_p[i] = p;
  }
}

// ===========================================================================
// Stage 2 (cont.): first own claim s_i of each request, and orphans.  A
// resident block past a request's first miss cannot be reached by lookup; it
// is dropped (invalidated) unless some request pinned it.
__global__ void __launch_bounds__(kWarpsPerCta * 32) k_claims(DevState s) {
  Ctl* c = s.ctl;
  if (c->status != PS_OK) return;
  if (c->hist_live + c->hist_new > s.history_capacity) {  // history capacity is sticky
    if (blockIdx.x == 0 && threadIdx.x == 0) { c->status = PS_ERR_CAPACITY; c->sticky = PS_ERR_CAPACITY; }
    return;
  }
  const int warp = threadIdx.x >> 5, lane = lane_id();
  const int i = blockIdx.x * kWarpsPerCta + warp;
  if (i >= s.R) return;
  const int n = s.rq_n[i], h = s.rq_h[i], pbase = s.rq_pbase[i];
  const uint32_t step32 = (uint32_t)c->step;
  int s_i = n;
  for (int c0 = h; c0 < n; c0 += 32) {
    const int m = c0 + lane;
    bool own = false;
    if (m < n) own = ldcg_u32(&s.claims[s.pos_claim[pbase + m]].minreq) == (uint32_t)i;
    const unsigned b = __ballot_sync(kFull, own);
    if (b) { s_i = c0 + __ffs(b) - 1; break; }
  }
  if (lane == 0) s.rq_s[i] = s_i;
  int ninv = 0;
  for (int c0 = h + 1; c0 < n; c0 += 32) {
    const int m = c0 + lane;
    bool inv = false;
    if (m < n) {
      const uint32_t b = s.pos_blk[pbase + m];
      if (b != kNone && ldcg_u32(s.blk_pin + b) != step32 && atomicExch(s.blk_inval + b, step32) != step32) {
        drop_block(s, b, PS_STAT_INVALIDATED_BLOCKS);
        atomicOr(s.bm_inval + (b >> 5), 1u << (b & 31));
        inv = true;
      }
    }
    ninv += __popc(__ballot_sync(kFull, inv));
  }
  if (lane == 0 && ninv) atomic_add_i64(&c->n_inval, ninv);
}

// ===========================================================================
// Stage 3: grant new blocks against the pool.  avail = free + unpinned
// resident = N - pinned; claims are ranked in (request, position) order; the
// first avail ranks are materialized.  One CTA.
__global__ void __launch_bounds__(1024) k_grant(DevState s) {
  Ctl* c = s.ctl;
  if (c->status != PS_OK) return;
  const int R = s.R;
  const int64_t avail = s.N - c->pinned;
  int32_t carry = 0;
  for (int t0 = 0; t0 < R; t0 += blockDim.x) {
    const int i = t0 + threadIdx.x;
    int32_t cl = 0;
    if (i < R) cl = s.rq_n[i] - s.rq_s[i];
    int32_t tot;
    const int32_t ex = block_excl_scan(cl, &tot);
    if (i < R) {
      const int64_t cb = carry + ex;
      s.rq_cbase[i] = (int32_t)cb;
      const int64_t a = tmin<int64_t>(cl, tmax<int64_t>(0, avail - cb));
      s.rq_a[i] = (int32_t)a;
      s.out.admitted_blocks[i] = (int32_t)a;
    }
    carry += tot;
  }
  const int64_t need = tmin<int64_t>(avail, carry);
  for (int i = threadIdx.x; i < R; i += blockDim.x) s.out.admitted_offsets[i] = (int32_t)tmin<int64_t>(s.rq_cbase[i], need);
  if (threadIdx.x == 0) {
    s.out.admitted_offsets[R] = (int32_t)need;
    const int64_t nfree = s.N - c->n_resident;
    c->avail = avail;
    c->total_claims = carry;
    c->need = need;
    c->nfree = nfree;
    c->ftake = min(need, nfree);
    c->mvict = need - min(need, nfree);
  }
}

// In-step hits: leading positions of [h_i, s_i) whose owner's claim was
// granted; hit_i = h_i + e_i.  Also records the first admitting request of
// each (group, prefix) entry.
__global__ void __launch_bounds__(kWarpsPerCta * 32) k_instep(DevState s) {
  Ctl* c = s.ctl;
  if (c->status != PS_OK) return;
  const int warp = threadIdx.x >> 5, lane = lane_id();
  const int i = blockIdx.x * kWarpsPerCta + warp;
  if (i >= s.R) return;
  const int h = s.rq_h[i], si = s.rq_s[i], pbase = s.rq_pbase[i];
  const int64_t avail = c->avail;
  int e = si - h;
  for (int c0 = h; c0 < si; c0 += 32) {
    const int m = c0 + lane;
    bool ungranted = false;
    if (m < si) {
      const uint32_t j = s.claims[s.pos_claim[pbase + m]].minreq;
      const int64_t rank = (int64_t)s.rq_cbase[j] + (m - s.rq_s[j]);
      ungranted = rank >= avail;
    }
    const unsigned b = __ballot_sync(kFull, ungranted);
    if (b) { e = c0 + __ffs(b) - 1 - h; break; }
  }
  if (lane == 0) {
    s.rq_e[i] = e;
    s.out.hit_blocks[i] = h + e;
    const uint32_t hs = s.rq_hs[i];
    if (s.rq_a[i] > 0 && hs != kNone)
      atomicMax(reinterpret_cast<unsigned long long*>(&s.hist[hs].atag), (unsigned long long)step_tag(c->step, (uint32_t)i));
  }
}

// ===========================================================================
// Stages 3-4: metering (Eq. 1-3, OnCacheFullBlocks of Alg. 1), in request
// order, one CTA per group.  Block-wide exclusive scans give each request the
// charges of the earlier requests of its group per contract, hence
//   D_g before the request (the gate of OnTouch, Eq. 4),
//   B_{g,c} after the request's own charge (the class of its new blocks).
// q_r >= 1 and "(g,p) was admitted" come from the history entry as it stood at
// the start of the step and the first request of the step that referenced /
// admitted it.  Also writes the group's statistics, balances and debts.
__global__ void __launch_bounds__(1024) k_meter(DevState s) {
  Ctl* c = s.ctl;
  if (c->status != PS_OK) return;
  const int g = blockIdx.x;
  const int C = s.C;
  const int64_t unit = (int64_t)1 << s.fp_shift;
  const uint64_t step = c->step;
  __shared__ int64_t B0[PS_MAX_CONTRACTS];
  if (threadIdx.x < C) {
    const int cc = threadIdx.x;
    B0[cc] = refill(s.ledger[g * C + cc], s.beta[cc], s.rho[cc], s.now - c->t_prev);
  }
  __syncthreads();
  int64_t carry[PS_MAX_CONTRACTS];
#pragma unroll
  for (int cc = 0; cc < PS_MAX_CONTRACTS; ++cc) carry[cc] = 0;
  int64_t st_req = 0, st_ptok = 0, st_full = 0, st_hit = 0, st_inst = 0, st_adm = 0, st_ungr = 0;
  const int R = s.R;
  for (int t0 = 0; t0 < R; t0 += blockDim.x) {
    const int i = t0 + threadIdx.x;
    const bool member = i < R && s.in_group[i] == g;
    int n = 0, a = 0, cid = 0;
    if (member) { n = s.rq_n[i]; a = s.rq_a[i]; cid = s.rq_cid[i]; }
    const bool pol = member && n > 0;
    int64_t S[PS_MAX_CONTRACTS];
#pragma unroll
    for (int cc = 0; cc < PS_MAX_CONTRACTS; ++cc) {
      if (cc < C) {
        int64_t tot;
        const int64_t ex = block_excl_scan<int64_t>((pol && cid == cc) ? a : 0, &tot);
        S[cc] = carry[cc] + ex;
        carry[cc] += tot;
      } else {
        S[cc] = 0;
      }
    }
    if (pol) {
      int64_t d = 0;
      for (int cc = 0; cc < C; ++cc) d += tmax<int64_t>(0, -(B0[cc] - S[cc] * unit));
      const bool gate = (s.flags & PS_FLAG_NO_DEBT_GATE) || d <= s.eps;
      const int64_t b_after = B0[cid] - (S[cid] + a) * unit;
      const uint32_t hs = s.rq_hs[i];
      HistEntry he{};
      if (hs != kNone) he = s.hist[hs];
      const uint32_t refadm = he.refadm;
      const bool q_ge1 = (refadm & 0x7FFFFFFFu) >= 1 || tag_req(he.ftag, step) < (uint32_t)i;
      const bool adm_before = (refadm >> 31) || tag_req(he.atag, step) < (uint32_t)i;
      const bool proven = q_ge1 && adm_before;
      s.rq_flags[i] = (uint8_t)((proven ? 1 : 0) | (gate ? 2 : 0));
      s.rq_knew[i] = (uint8_t)((b_after < -s.eps || !adm_before) ? kProb : kNormal);
      const int h = s.rq_h[i], e = s.rq_e[i];
      st_full += n; st_hit += h + e; st_inst += e; st_adm += a; st_ungr += (n - s.rq_s[i]) - a;
    }
    if (member) { st_req += 1; st_ptok += s.in_offsets[i + 1] - s.in_offsets[i]; }
  }
  st_req = block_sum(st_req); st_ptok = block_sum(st_ptok); st_full = block_sum(st_full);
  st_hit = block_sum(st_hit); st_inst = block_sum(st_inst); st_adm = block_sum(st_adm); st_ungr = block_sum(st_ungr);
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
    int64_t raw = 0, norm = 0, rmax = 0;
    for (int cc = 0; cc < C; ++cc) {
      const int64_t b = B0[cc] - carry[cc] * unit;  // Eq. 2 over the step's charges
      s.ledger[g * C + cc] = b;
      const int64_t def = tmax<int64_t>(0, -b);
      raw += def;                                    // Eq. 3
      norm += muldiv(def, s.rho_min, s.rho[cc]);     // Eq. 5
      if (b < 0) rmax = max(rmax, s.rho[cc]);
    }
    row[PS_STAT_DEBT_RAW] = raw;
    row[PS_STAT_DEBT_NORM] = norm;
    s.out.debt_raw[g] = raw;
    s.out.debt_norm[g] = norm;
    s.grp_P[g] = norm;
    s.grp_delta[g] = rmax ? muldiv(unit, s.rho_min, rmax) : 0;  // 1/W_g of Eq. 8
    s.grp_qsize[g] = 0;
  }
}

// ===========================================================================
// Stage 4: OnTouch (Alg. 1, Eq. 4) for every hit block, resident or in-step.
// Pass 1 applies the access updates (stamp = max, access count, S3-FIFO
// frequency) and records, per block, the lowest request whose touch promotes
// it.  Pass 2 counts the gated touches that precede the promotion (or all of
// them when none promotes) and applies the promotion of resident blocks.
__global__ void __launch_bounds__(kWarpsPerCta * 32) k_touch(DevState s) {
  Ctl* c = s.ctl;
  if (c->status != PS_OK) return;
  const int warp = threadIdx.x >> 5, lane = lane_id();
  const int i = blockIdx.x * kWarpsPerCta + warp;
  if (i >= s.R) return;
  const int n = s.rq_n[i];
  if (n == 0) return;
  const int h = s.rq_h[i], hit = h + s.rq_e[i], pbase = s.rq_pbase[i];
  const uint8_t fl = s.rq_flags[i];
  const bool proven = fl & 1, gate = fl & 2;
  const int cid = s.rq_cid[i];
  const uint64_t p = s.rq_p[i];
  const uint64_t step = c->step;
  for (int m = lane; m < hit; m += 32) {
    const int pos = pbase + m;
    bool elig;
    if (m < h) {
      const uint32_t b = s.pos_blk[pos];
      atomicMax(reinterpret_cast<unsigned long long*>(s.blk_stamp + b), (unsigned long long)make_stamp(step, i, m));
      atomicAdd(s.blk_acc + b, 1u);
      atomicAdd(s.blk_freq + b, 1u);
      elig = proven && s.blk_contract[b] == cid && s.blk_prefix[b] == p && s.blk_klass[b] != kReuse;
      if (elig && gate)
        atomicMax(reinterpret_cast<unsigned long long*>(s.blk_promo + b), (unsigned long long)step_tag(step, (uint32_t)i));
    } else {
      ClaimEntry* e = s.claims + s.pos_claim[pos];
      const uint32_t j = e->minreq;
      atomicMax(&e->last, (uint32_t)i + 1);
      atomicAdd(&e->tcnt, 1u);
      elig = proven && s.rq_cid[j] == cid && s.rq_p[j] == p;  // new blocks are never Reuse yet
      if (elig && gate) atomicMin(&e->promo, (uint32_t)i);
    }
    s.pos_elig[pos] = elig;
  }
}

__global__ void __launch_bounds__(kWarpsPerCta * 32) k_touch2(DevState s) {
  Ctl* c = s.ctl;
  if (c->status != PS_OK) return;
  const int warp = threadIdx.x >> 5, lane = lane_id();
  const int i = blockIdx.x * kWarpsPerCta + warp;
  if (i >= s.R) return;
  const int n = s.rq_n[i];
  if (n == 0) return;
  const int h = s.rq_h[i], hit = h + s.rq_e[i], pbase = s.rq_pbase[i];
  const bool gate = s.rq_flags[i] & 2;
  const uint64_t step = c->step;
  int gated = 0, promoted = 0;
  for (int m = lane; m < hit; m += 32) {
    const int pos = pbase + m;
    if (!s.pos_elig[pos]) continue;
    uint32_t promoter;
    uint32_t b = kNone;
    if (m < h) {
      b = s.pos_blk[pos];
      promoter = tag_req(ldcg_u64(s.blk_promo + b), step);
    } else {
      promoter = ldcg_u32(&s.claims[s.pos_claim[pos]].promo);
    }
    if (!gate) {
      if ((uint32_t)i < promoter) ++gated;
    } else if ((uint32_t)i == promoter) {
      ++promoted;
      if (b != kNone) s.blk_klass[b] = kReuse;
    }
  }
  gated = warp_sum(gated);
  promoted = warp_sum(promoted);
  if (lane == 0) {
    const int g = s.in_group[i];
    if (gated) atomic_add_i64(&stat_ref(s, g, PS_STAT_GATED_REUSES), gated);
    if (promoted) atomic_add_i64(&stat_ref(s, g, PS_STAT_PROMOTIONS), promoted);
  }
}

// ===========================================================================
// Stage 5: reclamation.  Candidates are resident blocks not hit in this step.
// The order key is (class, stamp) for prefixshield (Eq. 9; stamp only with
// the no-segmentation ablation) and the stamp for lru.
__global__ void k_cand(DevState s) {
  Ctl* c = s.ctl;
  if (c->status != PS_OK || c->mvict == 0) return;
  const uint32_t step32 = (uint32_t)c->step;
  const bool seg = s.policy == PS_PREFIXSHIELD && !(s.flags & PS_FLAG_NO_SEGMENTATION);
  for (int64_t b0 = blockIdx.x * (int64_t)blockDim.x; b0 < s.N; b0 += (int64_t)gridDim.x * blockDim.x) {
    const int64_t b = b0 + threadIdx.x;
    bool cand = false;
    uint32_t g = 0;
    if (b < s.N) {
      cand = (s.blk_flags[b] & 1) && s.blk_pin[b] != step32;
      uint64_t key = ~0ull;
      if (cand) {
        key = s.blk_stamp[b];
        if (seg) key |= (uint64_t)s.blk_klass[b] << 62;
        g = s.blk_group[b];
      }
      s.csk[b] = key;
    }
    if (s.policy == PS_PREFIXSHIELD) {
      const unsigned act = __ballot_sync(kFull, cand);
      if (cand) {
        const unsigned peers = __match_any_sync(act, g);
        if (lane_id() == __ffs(peers) - 1) atomic_add_i64(s.grp_qsize + g, __popc(peers));
      }
    }
  }
}

__global__ void k_sel_single(DevState s, int fallback) {
  Ctl* c = s.ctl;
  if (threadIdx.x != 0) return;
  int64_t m = 0;
  if (c->status == PS_OK) m = fallback ? c->m_fb : c->mvict;
  SelSeg z{};
  z.rank = m;
  z.active = m > 0;
  z.incl = 1;
  s.sel[0] = z;
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
__global__ void __launch_bounds__(1024) k_waterfill(DevState s) {
  Ctl* c = s.ctl;
  __shared__ int64_t s_tau;
  const int G = s.G;
  const int64_t eps = s.eps;
  const int64_t m = (c->status == PS_OK) ? c->mvict : 0;
  if (m == 0) {
    for (int g = threadIdx.x; g < G; g += blockDim.x) { s.sel[g].active = 0; s.grp_x[g] = 0; }
    if (threadIdx.x == 0) c->m_fb = 0;
    return;
  }
  // count of items with value > t, summed over groups
  auto count_gt = [&](int64_t t) -> int64_t {
    int64_t tot = 0;
    for (int g = threadIdx.x; g < G; g += blockDim.x) {
      const int64_t P = s.grp_P[g], d = s.grp_delta[g], q = s.grp_qsize[g];
      if (P > t && d > 0) tot += tmin<int64_t>(q, (P - t - 1) / d + 1);
    }
    return block_sum(tot);
  };
  const int64_t E = count_gt(eps);
  if (E <= m) {
    for (int g = threadIdx.x; g < G; g += blockDim.x) {
      const int64_t P = s.grp_P[g], d = s.grp_delta[g], q = s.grp_qsize[g];
      const int64_t x = (P > eps && d > 0) ? tmin<int64_t>(q, (P - eps - 1) / d + 1) : 0;
      s.grp_x[g] = x;
      SelSeg z{};
      z.rank = x; z.active = x > 0; z.incl = 1;
      s.sel[g] = z;
    }
    if (threadIdx.x == 0) { c->m_fb = m - E; c->sel_ntie = 0; c->sel_k = 0; }
    return;
  }
  // tau = max{t > eps : count_gt(t - 1) >= m}; binary search on [eps + 1, max P]
  int64_t pmax = 0;
  for (int g = threadIdx.x; g < G; g += blockDim.x) pmax = max(pmax, s.grp_P[g]);
  {
    __shared__ int64_t red[32];
    int64_t v = pmax;
    for (int o = 16; o > 0; o >>= 1) v = max(v, __shfl_xor_sync(kFull, v, o));
    if (lane_id() == 0) red[threadIdx.x >> 5] = v;
    __syncthreads();
    if (threadIdx.x == 0) {
      int64_t r = 0;
      for (int w = 0; w < (int)(blockDim.x >> 5); ++w) r = max(r, red[w]);
      s_tau = r;
    }
    __syncthreads();
    pmax = s_tau;
    __syncthreads();
  }
  int64_t lo = eps + 1, hi = pmax;  // invariant: count_gt(lo - 1) >= m
  while (lo < hi) {
    const int64_t mid = lo + (hi - lo + 1) / 2;
    if (count_gt(mid - 1) >= m) lo = mid; else hi = mid - 1;
  }
  const int64_t tau = lo;
  int64_t above = 0, ntie = 0;
  for (int g = threadIdx.x; g < G; g += blockDim.x) {
    const int64_t P = s.grp_P[g], d = s.grp_delta[g], q = s.grp_qsize[g];
    int64_t xa = 0;
    bool tied = false;
    if (P > tau && d > 0) xa = tmin<int64_t>(q, (P - tau - 1) / d + 1);
    if (d > 0 && P >= tau && (P - tau) % d == 0 && (P - tau) / d < q) tied = true;
    above += xa;
    ntie += tied;
    SelSeg z{};
    z.rank = xa + (tied ? 1 : 0);
    z.active = z.rank > 0;
    z.incl = tied ? 2 : 1;  // 2: the tie item is taken only if k_tie chooses it
    s.sel[g] = z;
    s.grp_x[g] = xa + (tied ? 1 : 0);
  }
  above = block_sum(above);
  ntie = block_sum(ntie);
  if (threadIdx.x == 0) {
    c->m_fb = 0;
    c->sel_ntie = (int32_t)ntie;
    c->sel_k = (int32_t)(m - above);  // tied items to take, 1..ntie
  }
}

// One MSB-first radix digit of the segmented select.  Every candidate of an
// active segment whose key matches the segment's prefix adds to that
// segment's histogram of the next 8-bit digit; the last CTA to finish picks,
// for every segment, the digit whose cumulative count reaches the rank.
__global__ void __launch_bounds__(256) k_radix_pass(DevState s, int pass, int single, int fallback) {
  Ctl* c = s.ctl;
  if (c->status != PS_OK || c->mvict == 0) return;
  const int nseg = single ? 1 : s.G;
  if (single && !s.sel[0].active) return;
  const int shift = 64 - kRadixBits * (pass + 1);
  for (int64_t b0 = blockIdx.x * (int64_t)blockDim.x; b0 < s.N; b0 += (int64_t)gridDim.x * blockDim.x) {
    const int64_t b = b0 + threadIdx.x;
    bool act = false;
    uint32_t idx = 0;
    if (b < s.N) {
      const uint64_t key = s.csk[b];
      if (key != ~0ull && !(fallback && ((s.bm_victim[b >> 5] >> (b & 31)) & 1))) {
        const int seg = single ? 0 : s.blk_group[b];
        const SelSeg ss = s.sel[seg];
        if (ss.active && (key & ss.mask) == ss.prefix) {
          act = true;
          idx = (uint32_t)seg * kRadixBins + (uint32_t)((key >> shift) & (kRadixBins - 1));
        }
      }
    }
    agg_inc(s.hist_bins, idx, act);
  }
  __shared__ bool last;
  __threadfence();
  __syncthreads();
  if (threadIdx.x == 0) last = atomicAdd(&c->ticket, 1u) == gridDim.x - 1;
  __syncthreads();
  if (!last) return;
  __threadfence();
  const int warp = threadIdx.x >> 5, lane = lane_id();
  for (int seg = warp; seg < nseg; seg += blockDim.x >> 5) {
    SelSeg ss = s.sel[seg];
    if (!ss.active) continue;
    uint32_t* row = s.hist_bins + (size_t)seg * kRadixBins;
    uint32_t v[kRadixBins / 32];
    uint32_t sum = 0;
#pragma unroll
    for (int j = 0; j < kRadixBins / 32; ++j) { v[j] = ldcg_u32(row + lane * (kRadixBins / 32) + j); sum += v[j]; }
    const uint32_t incl = warp_incl_scan(sum);
    const uint32_t excl = incl - sum;
    // the lane whose range holds the rank-th item
    const bool here = excl < (uint64_t)ss.rank && (uint64_t)ss.rank <= incl;
    const unsigned who = __ballot_sync(kFull, here);
    if (here) {
      uint32_t run = excl;
      int d = 0;
      for (int j = 0; j < kRadixBins / 32; ++j) {
        if ((uint64_t)ss.rank <= run + v[j]) { d = lane * (kRadixBins / 32) + j; break; }
        run += v[j];
      }
      ss.prefix |= (uint64_t)d << shift;
      ss.mask |= (uint64_t)(kRadixBins - 1) << shift;
      ss.rank -= run;
      s.sel[seg] = ss;
    }
    (void)who;
#pragma unroll
    for (int j = 0; j < kRadixBins / 32; ++j) row[lane * (kRadixBins / 32) + j] = 0;
  }
  if (threadIdx.x == 0) c->ticket = 0;
}

// Ties at tau (Eq. 7's tie rule: equal projected debt is broken by the
// retention segment and native queue order of each group's next candidate):
// among the groups holding an item at exactly tau (incl == 2 after the
// water-filling), the k with the smallest candidate keys take it.
__global__ void __launch_bounds__(1024) k_tie(DevState s) {
  Ctl* c = s.ctl;
  if (c->status != PS_OK || c->mvict == 0 || c->sel_ntie == 0) return;
  const int G = s.G;
  const int64_t k = c->sel_k;
  __shared__ uint64_t tkey[PS_MAX_GROUPS];
  __shared__ int tied[PS_MAX_GROUPS];
  for (int g = threadIdx.x; g < G; g += blockDim.x) {
    const SelSeg sg = s.sel[g];
    tied[g] = sg.active && sg.incl == 2;
    tkey[g] = sg.prefix;
  }
  __syncthreads();
  for (int g = threadIdx.x; g < G; g += blockDim.x) {
    if (!tied[g]) continue;
    int rank = 0;
    for (int h = 0; h < G; ++h) rank += tied[h] && tkey[h] < tkey[g];
    const bool chosen = rank < k;
    s.sel[g].incl = chosen ? 1 : 0;
    if (!chosen) s.grp_x[g] -= 1;
  }
}

// Mark victims: keys below (or equal to, if incl) the located threshold.
__global__ void k_mark(DevState s, int single, int fallback) {
  Ctl* c = s.ctl;
  if (c->status != PS_OK || c->mvict == 0) return;
  if (single && !s.sel[0].active) return;
  int marked = 0;
  for (int64_t b0 = blockIdx.x * (int64_t)blockDim.x; b0 < s.N; b0 += (int64_t)gridDim.x * blockDim.x) {
    const int64_t b = b0 + threadIdx.x;
    bool v = false;
    if (b < s.N) {
      const uint64_t key = s.csk[b];
      if (key != ~0ull && !(fallback && ((s.bm_victim[b >> 5] >> (b & 31)) & 1))) {
        const SelSeg ss = s.sel[single ? 0 : s.blk_group[b]];
        v = ss.active && (key < ss.prefix || (ss.incl && key == ss.prefix));
      }
    }
    const unsigned bits = __ballot_sync(kFull, v);
    if (bits && lane_id() == 0) {
      // 32 consecutive block ids share one bitmap word when b0 is 32-aligned
      atomicOr(s.bm_victim + ((b - lane_id()) >> 5), bits);
    }
    marked += __popc(bits);
  }
  if (lane_id() == 0 && marked) atomic_add_i64(&c->n_victims_marked, marked);
}

// TakeTrueFree (Alg. 2): the ftake smallest free block ids, plus the victims,
// form the allocated set (one CTA, contiguous word ranges per thread).
__global__ void __launch_bounds__(1024) k_freetake(DevState s) {
  Ctl* c = s.ctl;
  if (c->status != PS_OK) return;
  const int64_t ftake = c->ftake;
  const int64_t nw = s.nwords;
  const int64_t per = (nw + blockDim.x - 1) / blockDim.x;
  const int64_t w0 = tmin<int64_t>(nw, threadIdx.x * per), w1 = tmin<int64_t>(nw, w0 + per);
  auto free_word = [&](int64_t w) -> uint32_t {
    uint32_t f = ~s.res_bits[w];
    const int64_t hi = (w + 1) * 32;
    if (hi > s.N) f &= (1u << (uint32_t)(32 - (hi - s.N))) - 1u;
    return f;
  };
  int64_t cnt = 0;
  if (ftake > 0)
    for (int64_t w = w0; w < w1; ++w) cnt += __popc(free_word(w));
  int64_t tot;
  int64_t before = block_excl_scan(cnt, &tot);
  for (int64_t w = w0; w < w1; ++w) {
    uint32_t take = 0;
    if (ftake > 0 && before < ftake) {
      uint32_t f = free_word(w);
      while (f && before < ftake) {
        const uint32_t lsb = f & (0u - f);
        take |= lsb;
        f ^= lsb;
        ++before;
      }
    }
    s.bm_alloc[w] = take | s.bm_victim[w];
  }
}

// Evict the victims: drop their table entries and metadata.
__global__ void k_evict(DevState s) {
  Ctl* c = s.ctl;
  if (c->status != PS_OK || c->mvict == 0) return;
  for (int64_t w = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; w < s.nwords; w += (int64_t)gridDim.x * blockDim.x) {
    uint32_t bits = s.bm_victim[w];
    while (bits) {
      const int j = __ffs(bits) - 1;
      bits &= bits - 1;
      drop_block(s, (uint32_t)(w * 32 + j), PS_STAT_EVICTED_BLOCKS);
    }
  }
}

// Bitmaps -> ascending id lists (allocated, evicted, invalidated).  Each CTA
// owns 1024 bitmap words; pass 1 counts, pass 2 scans the counts and writes.
constexpr int kBmChunk = 1024;
__global__ void __launch_bounds__(1024) k_bm_count(DevState s) {
  if (s.ctl->status != PS_OK) return;
  const int64_t w = (int64_t)blockIdx.x * kBmChunk + threadIdx.x;
  const uint32_t* bms[3] = {s.bm_alloc, s.bm_victim, s.bm_inval};
  const int nchunks = gridDim.x;
  for (int k = 0; k < 3; ++k) {
    const int v = w < s.nwords ? __popc(bms[k][w]) : 0;
    const int t = block_sum(v);
    if (threadIdx.x == 0) s.bm_chunk_cnt[k * nchunks + blockIdx.x] = t;
  }
}
__global__ void __launch_bounds__(1024) k_bm_write(DevState s) {
  if (s.ctl->status != PS_OK) return;
  const int64_t w = (int64_t)blockIdx.x * kBmChunk + threadIdx.x;
  uint32_t* bms[3] = {s.bm_alloc, s.bm_victim, s.bm_inval};
  int32_t* outs[3] = {s.out.admitted_ids, s.out.evicted_ids, s.out.invalidated_ids};
  const int nchunks = gridDim.x;
  for (int k = 0; k < 3; ++k) {
    int base = 0;
    for (int j = threadIdx.x; j < blockIdx.x; j += blockDim.x) base += s.bm_chunk_cnt[k * nchunks + j];
    base = block_sum(base);
    const uint32_t bits = w < s.nwords ? bms[k][w] : 0u;
    int tot;
    const int ex = block_excl_scan(__popc(bits), &tot);
    int o = base + ex;
    uint32_t b = bits;
    while (b) {
      const int j = __ffs(b) - 1;
      b &= b - 1;
      if (o < s.max_blocks) outs[k][o] = (int32_t)(w * 32 + j);
      ++o;
    }
    if (w < s.nwords) bms[k][w] = 0;
    if (blockIdx.x == nchunks - 1 && threadIdx.x == 0) {
      if (k == 0) s.ctl->n_alloc = base + tot;
      if (k == 1) s.ctl->n_evicted = base + tot;
    }
  }
}

// Stage 6: place granted claims.  The allocated ids (ascending) go to the
// granted keys in (request, position) order; each new block carries the
// metadata OnCacheFullBlocks attached plus any in-step touches.
__global__ void __launch_bounds__(kWarpsPerCta * 32) k_insert(DevState s) {
  Ctl* c = s.ctl;
  if (c->status != PS_OK) return;
  const int warp = threadIdx.x >> 5, lane = lane_id();
  const int i = blockIdx.x * kWarpsPerCta + warp;
  if (i >= s.R) return;
  const int a = s.rq_a[i];
  if (a == 0) return;
  const int si = s.rq_s[i], pbase = s.rq_pbase[i], cb = s.rq_cbase[i];
  const uint32_t g = (uint32_t)s.in_group[i];
  const uint8_t cid = (uint8_t)s.rq_cid[i];
  const uint64_t p = s.rq_p[i];
  const uint8_t knew = s.rq_knew[i];
  const uint64_t step = c->step;
  const int64_t n_alloc = c->n_alloc;
  bool bad = false;
  for (int m = si + lane; m < si + a; m += 32) {
    const int pos = pbase + m;
    if (cb + (m - si) >= n_alloc) { bad = true; continue; }  // allocated set short: internal error
    const uint32_t b = (uint32_t)s.out.admitted_ids[cb + (m - si)];
    if (b >= (uint64_t)s.N) { bad = true; continue; }
    const ClaimEntry e = s.claims[s.pos_claim[pos]];
    const uint64_t key = s.pos_key[pos];
    s.blk_key[b] = key;
    s.blk_group[b] = (uint16_t)g;
    s.blk_contract[b] = cid;
    s.blk_prefix[b] = p;
    s.blk_klass[b] = e.promo != kNone ? (uint8_t)kReuse : knew;
    s.blk_stamp[b] = make_stamp(step, e.last ? e.last - 1 : (uint32_t)i, m);
    s.blk_acc[b] = e.tcnt;
    s.blk_freq[b] = e.tcnt;
    s.blk_flags[b] = 1;
    s.blk_slot[b] = table_insert(s, key, g, b);
    atomicOr(s.res_bits + (b >> 5), 1u << (b & 31));
  }
  if (__any_sync(kFull, bad) && lane == 0) c->internal_error = 1;
  if (lane == 0) {
    atomic_add_i64(&c->n_resident, a);
    atomic_add_i64(&stat_ref(s, g, PS_STAT_RESIDENT_BLOCKS), a);
  }
}

// OnRequest / RecordSuccessfulAdmission commit: reference counts and admitted
// flags of the history entries.
__global__ void k_hist_commit(DevState s) {
  Ctl* c = s.ctl;
  if (c->status != PS_OK) return;
  const int i = blockIdx.x * blockDim.x + threadIdx.x;
  if (i == 0) c->hist_live += c->hist_new;
  if (i >= s.R || s.rq_n[i] == 0) return;
  const uint32_t hs = s.rq_hs[i];
  if (hs == kNone) return;
  atomicAdd(&s.hist[hs].refadm, 1u);
  if (s.rq_a[i] > 0) atomicOr(&s.hist[hs].refadm, 0x80000000u);
}

// Clear the claim-map slots this step used.
__global__ void __launch_bounds__(kWarpsPerCta * 32) k_claim_clear(DevState s) {
  Ctl* c = s.ctl;
  if (c->status != PS_OK) return;
  const int warp = threadIdx.x >> 5, lane = lane_id();
  const int i = blockIdx.x * kWarpsPerCta + warp;
  if (i >= s.R) return;
  const int n = s.rq_n[i], h = s.rq_h[i], pbase = s.rq_pbase[i];
  for (int m = h + lane; m < n; m += 32) {
    const uint32_t slot = s.pos_claim[pbase + m];
    if (slot == kNone) continue;
    ClaimEntry z{};
    z.key = 0; z.minreq = kNone; z.last = 0; z.tcnt = 0; z.promo = kNone; z.pad0 = 0; z.pad1 = 0;
    s.claims[slot] = z;
  }
}

__global__ void k_finalize(DevState s) {
  Ctl* c = s.ctl;
  if (threadIdx.x != 0 || blockIdx.x != 0) return;
  const int32_t st = c->internal_error ? PS_ERR_DEVICE_STATUS : c->status;
  s.out.counts[3] = st;
  if (st != PS_OK) return;
  s.out.counts[0] = (int32_t)c->need;
  s.out.counts[1] = (int32_t)c->n_evicted;
  s.out.counts[2] = (int32_t)c->n_inval;
  c->t_prev = s.now;
  c->step += 1;
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
  k_init_blocks<<<grid_for(s.N, 256, 152 * 8), 256, 0, st>>>(s);
  k_init_ctl<<<1, 1024, 0, st>>>(s);
}

template <int PPB>
static void launch_hash(const DevState& s, cudaStream_t st) {
  const size_t smem = (size_t)kWarpsPerCta * (32 * 2 * PPB + 4) * sizeof(int32_t);
  static bool configured = false;
  if (!configured) {
    cudaFuncSetAttribute(k_hash_lookup<PPB>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    configured = true;
  }
  k_hash_lookup<PPB><<<(s.R + kWarpsPerCta - 1) / kWarpsPerCta, kWarpsPerCta * 32, smem, st>>>(s);
}

int32_t launch_step(const DevState& s, cudaStream_t st, StepTrace* tr) {
  const int R = s.R;
  const int wgrid = R > 0 ? (R + kWarpsPerCta - 1) / kWarpsPerCta : 1;
  const int wthreads = kWarpsPerCta * 32;
  const int ngrid = grid_for(s.N, 256, 152 * 8);
  int launches = 0;
  auto mark = [&](int stage) {
    if (tr && tr->timing) cudaEventRecord(tr->ev[stage], st);
  };
#define PS_LAUNCH(...) do { __VA_ARGS__; ++launches; } while (0)
  mark(0);
  PS_LAUNCH(k_validate<<<1, 1024, 0, st>>>(s));
  mark(1);
  if (R > 0) {
    switch (s.bs / 2) {
      case 1: PS_LAUNCH(launch_hash<1>(s, st)); break;
      case 2: PS_LAUNCH(launch_hash<2>(s, st)); break;
      case 4: PS_LAUNCH(launch_hash<4>(s, st)); break;
      case 8: PS_LAUNCH(launch_hash<8>(s, st)); break;
      case 16: PS_LAUNCH(launch_hash<16>(s, st)); break;
      case 32: PS_LAUNCH(launch_hash<32>(s, st)); break;
      default: return PS_ERR_INVALID_ARG;
    }
  }
  mark(2);
  PS_LAUNCH(k_claims<<<wgrid, wthreads, 0, st>>>(s));
  mark(3);
  PS_LAUNCH(k_grant<<<1, 1024, 0, st>>>(s));
  PS_LAUNCH(k_instep<<<wgrid, wthreads, 0, st>>>(s));
  mark(4);
  PS_LAUNCH(k_meter<<<s.G, 1024, 0, st>>>(s));
  mark(5);
  PS_LAUNCH(k_touch<<<wgrid, wthreads, 0, st>>>(s));
  PS_LAUNCH(k_touch2<<<wgrid, wthreads, 0, st>>>(s));
  mark(6);
  PS_LAUNCH(k_cand<<<ngrid, 256, 0, st>>>(s));
  if (s.policy == PS_PREFIXSHIELD) {
    PS_LAUNCH(k_waterfill<<<1, 1024, 0, st>>>(s));
    for (int pass = 0; pass < 8; ++pass) PS_LAUNCH(k_radix_pass<<<ngrid, 256, 0, st>>>(s, pass, 0, 0));
    PS_LAUNCH(k_tie<<<1, 1024, 0, st>>>(s));
    PS_LAUNCH(k_mark<<<ngrid, 256, 0, st>>>(s, 0, 0));
    PS_LAUNCH(k_sel_single<<<1, 32, 0, st>>>(s, 1));
    for (int pass = 0; pass < 8; ++pass) PS_LAUNCH(k_radix_pass<<<ngrid, 256, 0, st>>>(s, pass, 1, 1));
    PS_LAUNCH(k_mark<<<ngrid, 256, 0, st>>>(s, 1, 1));
  } else if (s.policy == PS_LRU) {
    PS_LAUNCH(k_sel_single<<<1, 32, 0, st>>>(s, 0));
    for (int pass = 0; pass < 8; ++pass) PS_LAUNCH(k_radix_pass<<<ngrid, 256, 0, st>>>(s, pass, 1, 0));
    PS_LAUNCH(k_mark<<<ngrid, 256, 0, st>>>(s, 1, 0));
  } else {
    return PS_ERR_INVALID_ARG;  // S3-FIFO: not yet
  }
  mark(7);
  PS_LAUNCH(k_freetake<<<1, 1024, 0, st>>>(s));
  PS_LAUNCH(k_evict<<<grid_for(s.nwords, 256, 152 * 4), 256, 0, st>>>(s));
  mark(8);
  const int nchunks = (int)((s.nwords + kBmChunk - 1) / kBmChunk);
  PS_LAUNCH(k_bm_count<<<nchunks, 1024, 0, st>>>(s));
  PS_LAUNCH(k_bm_write<<<nchunks, 1024, 0, st>>>(s));
  mark(9);
  PS_LAUNCH(k_insert<<<wgrid, wthreads, 0, st>>>(s));
  mark(10);
  PS_LAUNCH(k_hist_commit<<<grid_for(R, 256, 1 << 20), 256, 0, st>>>(s));
  PS_LAUNCH(k_claim_clear<<<wgrid, wthreads, 0, st>>>(s));
  PS_LAUNCH(k_finalize<<<1, 32, 0, st>>>(s));
  mark(11);
#undef PS_LAUNCH
  if (tr) tr->launches = launches;
  return cudaGetLastError() == cudaSuccess ? PS_OK : PS_ERR_CUDA;
}

}  // namespace ps
