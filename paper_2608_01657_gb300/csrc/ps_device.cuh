// Device helpers shared by the step's kernel files: warp and CTA scans,
// warp-aggregated atomics, and cache-hinted loads.
#pragma once

#include "ps_internal.cuh"

namespace ps {

constexpr unsigned kFull = 0xFFFFFFFFu;
constexpr int kThreads = 256;     // position-parallel kernels

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
// Four exclusive scans in one pass: thread t holds the elements
// u * blockDim.x + t (u = 0..3) of a 4 * blockDim.x tile, so its loads stay
// coalesced; ex[u] receives the exclusive prefix of its element u in tile
// order, *total the tile's sum.  Two barriers for the whole tile.
template <typename T>
__device__ void block_excl_scan4(const T (&v)[4], T (&ex)[4], T* total) {
  __shared__ T wsum[4][32];
  const int lane = lane_id(), warp = threadIdx.x >> 5, nw = blockDim.x >> 5;
  T incl[4];
#pragma unroll
  for (int u = 0; u < 4; ++u) {
    incl[u] = warp_incl_scan(v[u]);
    if (lane == 31) wsum[u][warp] = incl[u];
  }
  __syncthreads();
  if (warp < 4) {  // warp u scans row u of the warp totals
    T w = lane < nw ? wsum[warp][lane] : T(0);
    T wi = warp_incl_scan(w);
    __syncwarp();
    wsum[warp][lane] = wi;
  }
  __syncthreads();
  T carry = T(0);
#pragma unroll
  for (int u = 0; u < 4; ++u) {
    ex[u] = carry + (warp ? wsum[u][warp - 1] : T(0)) + incl[u] - v[u];
    carry += wsum[u][nw - 1];
  }
  *total = carry;
  __syncthreads();
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
__device__ __forceinline__ int64_t* stat_ptr(const DevState& s, int g, int k) {
  return s.stats + (int64_t)g * PS_NUM_STATS + k;
}
// Add v to stat k of group g, combining lanes of the warp with equal g.
__device__ __forceinline__ void agg_stat(const DevState& s, uint32_t g, int k, int64_t v, bool active) {
  const bool on = active && v != 0;
  const unsigned act = __ballot_sync(kFull, on);
  if (!on) return;
  const unsigned peers = __match_any_sync(act, g);
  int64_t sum = 0;
  for (unsigned m = peers; m; m &= m - 1) sum += __shfl_sync(peers, v, __ffs(m) - 1);
  if (lane_id() == __ffs(peers) - 1) atomic_add_i64(stat_ptr(s, (int)g, k), sum);
}
// Warp-aggregated increment of bins[idx] for the lanes with 'active'.
__device__ __forceinline__ void agg_inc(uint32_t* bins, uint32_t idx, bool active) {
  const unsigned act = __ballot_sync(kFull, active);
  if (!active) return;
  const unsigned peers = __match_any_sync(act, idx);
  if (lane_id() == __ffs(peers) - 1) atomicAdd(bins + idx, (uint32_t)__popc(peers));
}
// base[i] += v, lanes of the warp with equal i combined first (every lane of
// the warp must call it).
__device__ __forceinline__ void agg_add_i64(int64_t* base, uint32_t i, int64_t v, bool active) {
  const unsigned act = __ballot_sync(kFull, active);
  if (!active) return;
  const unsigned peers = __match_any_sync(act, i);
  int64_t sum = 0;
  for (unsigned m = peers; m; m &= m - 1) sum += __shfl_sync(peers, v, __ffs(m) - 1);
  if (lane_id() == __ffs(peers) - 1) atomicAdd(reinterpret_cast<unsigned long long*>(base + i), (unsigned long long)sum);
}
// atomicMin of v into base[i], lanes of the warp with equal i combined first
// (every lane of the warp must call it).
__device__ __forceinline__ void agg_min_u32(uint32_t* base, uint32_t i, uint32_t v, bool active) {
  const unsigned act = __ballot_sync(kFull, active);
  if (!active) return;
  const unsigned peers = __match_any_sync(act, i);
  const uint32_t m = __reduce_min_sync(peers, v);
  if (lane_id() == __ffs(peers) - 1) atomicMin(base + i, m);
}
__device__ __forceinline__ uint64_t ldcg_u64(const uint64_t* p) { return __ldcg(reinterpret_cast<const unsigned long long*>(p)); }
__device__ __forceinline__ uint32_t ldcg_u32(const uint32_t* p) { return __ldcg(p); }

// ---- published words: a value and its flags in one aligned 64-bit word -----
// One relaxed 64-bit store publishes both, and one relaxed 64-bit load reads
// both, so no fence is needed to order them.
constexpr int kSpinLimit = 1 << 20;

__device__ __forceinline__ void st_relaxed_u64(uint64_t* p, uint64_t v) {
  asm volatile("st.relaxed.gpu.global.u64 [%0], %1;" ::"l"(p), "l"(v) : "memory");
}
__device__ __forceinline__ uint64_t ld_relaxed_u64(const uint64_t* p) {
  uint64_t v;
  asm volatile("ld.relaxed.gpu.global.u64 %0, [%1];" : "=l"(v) : "l"(p) : "memory");
  return v;
}
// Wait (bounded) until every bit of 'need' is set in *w; the word, or 0 if
// the wait ran out.
__device__ __forceinline__ uint64_t wait_word(const uint64_t* w, uint64_t need) {
  for (int it = 0; it < kSpinLimit; ++it) {
    const uint64_t v = ld_relaxed_u64(w);
    if ((v & need) == need) return v;
    __nanosleep(32);
  }
  return 0;
}

// ---- indexed queues: which logs hold a block ---------------------------------
__device__ __forceinline__ bool lg_segmented(const DevState& s) {
  return s.policy == PS_PREFIXSHIELD && !(s.flags & PS_FLAG_NO_SEGMENTATION);
}
// The per-group log (A) and the global log (B) of a block of group g and
// class k; -1 where the policy keeps no such log.
__device__ __forceinline__ int32_t lg_log_a(const DevState& s, uint32_t g, uint32_t k) {
  return s.policy == PS_LRU ? -1 : (int32_t)(g * kClasses + (lg_segmented(s) ? k : 0u));
}
__device__ __forceinline__ int32_t lg_log_b(const DevState& s, uint32_t k) {
  return s.policy == PS_STATICQUOTA ? -1 : (int32_t)((uint32_t)s.G * kClasses + (lg_segmented(s) ? k : 0u));
}

}  // namespace ps
