// S3-FIFO baseline (Yang, Zhang, Qiu, Yue, Vinayak, SOSP 2023), the paper's
// reuse-aware replacement baseline (Sec. V-A): a small FIFO (10% of the
// pool), a main FIFO, a ghost FIFO of evicted small-queue keys, and a capped
// frequency counter, with no tenant metadata.
//
// The published algorithm evicts one block at a time, each decision reading
// the state the previous one left.  A step's m evictions nevertheless have a
// closed form, which the kernels here compute with prefix counts:
//
//   - Small phase.  An eviction that takes the small queue pops its unpinned
//     members oldest first: a member with frequency >= the move threshold
//     goes to the main queue's head, the first one below it is the victim
//     (its key enters the ghost).  Eviction t takes the small queue while the
//     queue held at least its capacity when it started, i.e. while the
//     members popped before it number at most D = |small| - capacity, and an
//     unpinned member is left.  So the phase consumes a prefix of the small
//     queue's K unpinned members: up to its n_A-th victim,
//     n_A = min(m, 1 + #{victims among the first min(D, K - 1)}), or all of
//     them when it runs out of victims (that eviction then takes the main
//     queue).
//   - Main phase.  The remaining m_B evictions visit the main queue (its
//     unpinned members, then the moved blocks) from the tail: frequency f > 0
//     reinserts the block at the head with f - 1, f = 0 evicts it.  So the
//     visits go in rounds over that list, round r visiting the members with
//     f >= r in list order, and a member of frequency f leaves on its
//     (f + 1)-th visit.  The per-frequency counts fix the final round Rs and
//     the list position P of the last visit; every member's fate, new
//     frequency and new sequence number follow from its position and the
//     counts of members with f >= Rs and f > Rs before it.
//   - This holds while the main queue never runs empty (m_B at most the
//     list's length) and frequencies stay below kS3Bins.  Otherwise a
//     sequential kernel replays the published loop on the same arrays.
//
// Representation.  Each queue is an array of block ids in sequence order,
// oldest first (pinned blocks stay in place).  A step reads one buffer and
// writes the other: the small queue's kept members then the step's
// insertions; the main queue's kept members, the blocks the step moved or
// reinserted (in their new sequence order), then its insertions.  The ghost
// is a bucketed map (group, key) -> FIFO position, a sequence number per map
// slot, and a FIFO ring of map slots with a bitmap of live positions; a
// ghost hit clears its position, and pushes beyond the ghost's capacity trim
// the oldest live ones.  When the ring lacks room for a step's pushes, its
// live positions are compacted into the other ring.
#include "ps_device.cuh"
#include "ps_launch.cuh"

namespace ps {

namespace {

constexpr int kCT = 256;                // threads of the chunk kernels
constexpr int kPer = kS3Chunk / kCT;    // entries a thread
constexpr int kPT = 1024;               // threads of the planner
constexpr int kRingWords = kS3Chunk / 32;

__device__ __forceinline__ int64_t cdiv64(int64_t a, int64_t b) { return (a + b - 1) / b; }
__device__ __forceinline__ uint32_t* q_region(const DevState& s, int buf, int r) {
  return s.s3_arr + ((size_t)buf * 2 + (size_t)r) * (size_t)s.s3_np;
}
__device__ __forceinline__ uint32_t* ring_of(const DevState& s, int rb) {
  return s.ghost_ring + (size_t)rb * s.ghost_ring_cap;
}
__device__ __forceinline__ uint32_t* bits_of(const DevState& s, int rb) {
  return s.ghost_bits + (size_t)rb * (s.ghost_ring_cap / 32);
}
__device__ __forceinline__ uint32_t eff_freq(const DevState& s, uint32_t b) {
  const uint32_t f = s.blk_freq[b];
  return f < (uint32_t)s.s3_freq_cap ? f : (uint32_t)s.s3_freq_cap;
}
// A queue array write; a position past the region means the plan is
// inconsistent, which is reported instead of written.
__device__ __forceinline__ void q_put(const DevState& s, uint32_t* region, int64_t pos, uint32_t b) {
  if (pos >= 0 && pos < s.s3_np) region[pos] = b;
  else s.ctl->internal_error = 1;
}
__device__ __forceinline__ void mark_victim(const DevState& s, uint32_t b) {
  atomicOr(s.bm_victim + (b >> 5), 1u << (b & 31));
}

// ---- ghost map: 8-way buckets of {key, FIFO index, group} --------------------
// Lookup: the bucket's ways and overflow count in one round of loads.
__device__ uint32_t gh_find(const DevState& s, uint64_t key, uint32_t g) {
  const uint32_t mask = (1u << s.gh_nbuckets_log2) - 1;
  uint32_t b = table_home(key, g, s.gh_nbuckets_log2);
  for (uint32_t it = 0; it <= mask; ++it) {
    const uint4* e = reinterpret_cast<const uint4*>(s.ghost_map + (size_t)b * kTableWays);
    uint4 raw[kTableWays];
#pragma unroll
    for (int w = 0; w < kTableWays; ++w) raw[w] = __ldcg(e + w);
    const uint32_t ovf = __ldcg(s.ghost_ovf + b);
    uint32_t hit = kNone;
#pragma unroll
    for (int w = 0; w < kTableWays; ++w)
      if (raw[w].z != kNone && raw[w].x == (uint32_t)key && raw[w].y == (uint32_t)(key >> 32) && raw[w].w == g)
        hit = b * kTableWays + w;
    if (hit != kNone || ovf == 0) return hit;
    b = (b + 1) & mask;
  }
  return kNone;
}
// Insert (no key is in the map twice); a slot is taken by swapping its FIFO
// index in, then its key, group and sequence number are written.
__device__ uint32_t gh_insert(const DevState& s, uint64_t key, uint32_t g, uint32_t ridx, uint64_t seq) {
  const uint32_t mask = (1u << s.gh_nbuckets_log2) - 1;
  uint32_t b = table_home(key, g, s.gh_nbuckets_log2);
  const uint32_t w0 = (uint32_t)(key >> 7) & (kTableWays - 1);
  for (uint32_t it = 0; it <= mask; ++it) {
    TableEntry* e = s.ghost_map + (size_t)b * kTableWays;
    for (int q = 0; q < kTableWays; ++q) {
      const int w = (int)((w0 + (uint32_t)q) & (kTableWays - 1));
      if (atomicCAS(&e[w].blk, kNone, ridx) == kNone) {
        e[w].key = key;
        e[w].grp = g;
        const uint32_t slot = b * kTableWays + (uint32_t)w;
        s.ghost_sq[slot] = seq;
        return slot;
      }
    }
    atomicAdd(s.ghost_ovf + b, 1u);
    b = (b + 1) & mask;
  }
  return kNone;
}
// Release a slot whose key and group are known; the overflow counters of the
// buckets the key probed past are repaired.
__device__ void gh_erase_known(const DevState& s, uint32_t slot, uint64_t key, uint32_t g) {
  const uint32_t mask = (1u << s.gh_nbuckets_log2) - 1;
  s.ghost_map[slot].blk = kNone;
  const uint32_t bucket = slot / kTableWays;
  uint32_t x = table_home(key, g, s.gh_nbuckets_log2);
  for (uint32_t it = 0; x != bucket && it <= mask; ++it, x = (x + 1) & mask) atomicSub(s.ghost_ovf + x, 1u);
}
// Release a slot, reading its key and group first.  Erasures and insertions
// never run in the same kernel (a step's pushes are inserted by k_s3_push,
// after the trimming), so no other thread rewrites the slot meanwhile.
__device__ void gh_erase(const DevState& s, uint32_t slot) {
  const uint64_t key = __ldcg(reinterpret_cast<const unsigned long long*>(&s.ghost_map[slot].key));
  const uint32_t g = __ldcg(&s.ghost_map[slot].grp);
  gh_erase_known(s, slot, key, g);
}
// The step's small-queue victims in eviction order (their ghost pushes): the
// second half of the candidate-key scratch, which S3-FIFO does not use.
__device__ __forceinline__ uint32_t* push_list(const DevState& s) {
  return reinterpret_cast<uint32_t*>(s.csk) + s.N;
}

// A locate of the planner found nothing (never expected): the step goes to
// the sequential kernel and reports an internal error.  Every thread of the
// planner sees the same shared result, so all return together.
__device__ void lost_locate(const DevState& s) {
  if (threadIdx.x == 0) {
    s.s3_plan->fb = 1;
    s.ctl->internal_error = 1;
  }
}

// ---- block-wide helpers of the planner (kPT threads) ----------------------------
// Exclusive scan of n items, each thread a run of consecutive items: get(i)
// gives item i, put(i, excl, v) receives its exclusive prefix.  Returns the total.
template <typename Get, typename Put>
__device__ uint64_t plan_scan(int64_t n, Get get, Put put) {
  const int64_t per = (n + kPT - 1) / kPT;
  const int64_t i0 = (int64_t)threadIdx.x * per, i1 = tmin<int64_t>(n, i0 + per);
  uint64_t loc = 0;
  for (int64_t i = i0; i < i1; ++i) loc += get(i);
  uint64_t tot;
  uint64_t ex = block_excl_scan<uint64_t>(loc, &tot);
  for (int64_t i = i0; i < i1; ++i) {
    const uint64_t v = get(i);
    put(i, ex, v);
    ex += v;
  }
  __syncthreads();
  return tot;
}
// Inclusive scan over one chunk's entries (two a thread): val(j) gives the
// packed value of entry j (j < n), and at(j, incl, own) sees every entry.
template <typename Val, typename At>
__device__ void chunk_scan(int n, Val val, At at) {
  const int j0 = 2 * (int)threadIdx.x;
  const uint64_t v0 = j0 < n ? val(j0) : 0, v1 = j0 + 1 < n ? val(j0 + 1) : 0;
  uint64_t tot;
  const uint64_t ex = block_excl_scan<uint64_t>(v0 + v1, &tot);
  if (j0 < n) at(j0, ex + v0, v0);
  if (j0 + 1 < n) at(j0 + 1, ex + v0 + v1, v1);
  __syncthreads();
}

// entry attribute byte: bit0 live, bit1 unpinned (live and not hit this step), bits 4-7 frequency
__device__ __forceinline__ bool a_live(uint32_t a) { return a & 1; }
__device__ __forceinline__ bool a_un(uint32_t a) { return (a >> 1) & 1; }
__device__ __forceinline__ uint32_t a_f(uint32_t a) { return a >> 4; }

}  // namespace

// ===========================================================================
// 1. Per-chunk counts of both queues, each entry's attribute byte, and the
//    live ghost positions per ring chunk of the FIFO window.
__global__ void __launch_bounds__(kCT) k_s3_count(DevState s) {
  s = with_args(s);
  Ctl* c = s.ctl;
  if (c->status != PS_OK) return;
  const int buf = c->s3_buf;
  const int64_t len0 = c->s3_len[0], len1 = c->s3_len[1];
  const int64_t ch0 = cdiv64(len0, kS3Chunk), ch1 = cdiv64(len1, kS3Chunk);
  const uint64_t tail = c->ghost_tail, head = c->ghost_head;
  const uint64_t a0 = tail & ~(uint64_t)(kS3Chunk - 1);
  const int64_t nrch = head > tail ? cdiv64((int64_t)(head - a0), kS3Chunk) : 0;
  const uint32_t step32 = (uint32_t)c->step;
  const uint32_t cap = (uint32_t)s.s3_freq_cap, mm = (uint32_t)s.s3_move_min;
  const uint64_t rmask = s.ghost_ring_cap - 1;
  const uint32_t* rbits = bits_of(s, c->ghost_rbuf);
  // the insert kernels' per-chunk ghost-hit counters start at zero
  const int64_t nick = s.max_blocks / kS3Chunk + 1;
  for (int64_t i = blockIdx.x * (int64_t)kCT + threadIdx.x; i < nick; i += (int64_t)gridDim.x * kCT) s.s3_ick[i] = 0;
  __shared__ uint32_t sh[20];
  const int64_t units = ch0 + ch1 + nrch;
  for (int64_t u = blockIdx.x; u < units; u += gridDim.x) {
    if (threadIdx.x < 20) sh[threadIdx.x] = 0;
    __syncthreads();
    if (u < ch0 + ch1) {
      const int r = u < ch0 ? 0 : 1;
      const int64_t ci = r ? u - ch0 : u;
      const int64_t len = r ? len1 : len0;
      const int64_t j0 = ci * kS3Chunk + (int64_t)threadIdx.x * kPer;
      const uint4* ip = reinterpret_cast<const uint4*>(q_region(s, buf, r) + j0);
      const uint4 w0 = ip[0], w1 = ip[1];
      const uint32_t id[kPer] = {w0.x, w0.y, w0.z, w0.w, w1.x, w1.y, w1.z, w1.w};
      uint8_t fl[kPer];
      uint32_t pin[kPer], fr[kPer];
#pragma unroll
      for (int k = 0; k < kPer; ++k) {
        const bool v = j0 + k < len;
        fl[k] = v ? s.blk_flags[id[k]] : 0;
        pin[k] = v ? s.blk_pin[id[k]] : 0;
        fr[k] = v ? s.blk_freq[id[k]] : 0;
      }
      uint32_t nlive = 0, nu = 0, nev = 0;
      uint8_t a[kPer];
#pragma unroll
      for (int k = 0; k < kPer; ++k) {
        const bool live = j0 + k < len && (fl[k] & 1);
        const bool un = live && pin[k] != step32;
        const uint32_t f = tmin(fr[k], cap);
        const uint32_t fq = tmin(f, (uint32_t)(kS3Bins - 1));
        a[k] = (uint8_t)((live ? 1u : 0u) | (un ? 2u : 0u) | (fq << 4));
        nlive += live;
        nu += un;
        nev += un && f < mm;
        if (un) atomicAdd(&sh[4 + fq], 1u);
      }
      uint2 packed;
      packed.x = (uint32_t)a[0] | (uint32_t)a[1] << 8 | (uint32_t)a[2] << 16 | (uint32_t)a[3] << 24;
      packed.y = (uint32_t)a[4] | (uint32_t)a[5] << 8 | (uint32_t)a[6] << 16 | (uint32_t)a[7] << 24;
      *reinterpret_cast<uint2*>(s.s3_attr + (size_t)r * s.s3_np + j0) = packed;
      nlive = warp_sum(nlive);
      nu = warp_sum(nu);
      nev = warp_sum(nev);
      if (lane_id() == 0) {
        atomicAdd(&sh[0], nlive);
        atomicAdd(&sh[1], nu);
        atomicAdd(&sh[2], nev);
      }
      __syncthreads();
      if (threadIdx.x < 20) reinterpret_cast<uint32_t*>(s.s3_ck + (size_t)r * s.s3_nch + ci)[threadIdx.x] = sh[threadIdx.x];
    } else {
      const int64_t k = u - ch0 - ch1;
      const uint64_t p0 = a0 + (uint64_t)k * kS3Chunk;
      if (threadIdx.x < kRingWords) {
        const uint64_t pw = p0 + 32u * threadIdx.x;
        uint32_t w = rbits[(pw & rmask) >> 5];
        // positions outside [tail, head) do not count
        if (pw < tail) w = tail - pw >= 32 ? 0u : w & (~0u << (uint32_t)(tail - pw));
        if (pw + 32 > head) w = head <= pw ? 0u : w & (~0u >> (uint32_t)(pw + 32 - head));
        const uint32_t n = warp_sum((uint32_t)__popc(w));
        if (lane_id() == 0) atomicAdd(&sh[0], n);
      }
      __syncthreads();
      if (threadIdx.x == 0) s.s3_rck[k] = sh[0];
    }
  }
}

// ===========================================================================
// 2. The plan: one CTA turns the chunk counts into the step's closed form
//    (or hands the step to the sequential kernel), and every chunk's bases.
__global__ void __launch_bounds__(kPT) k_s3_plan(DevState s) {
  s = with_args(s);
  Ctl* c = s.ctl;
  if (c->status != PS_OK) return;
  S3Plan* pl = s.s3_plan;
  __shared__ int64_t sv[8];
  __shared__ uint32_t hmain[kS3Bins], hmov[kS3Bins];
  const int buf = c->s3_buf;
  const int64_t lenS = c->s3_len[0], lenM = c->s3_len[1];
  const int64_t chS = cdiv64(lenS, kS3Chunk), chM = cdiv64(lenM, kS3Chunk);
  const S3Chunk* ckS = s.s3_ck;
  const S3Chunk* ckM = s.s3_ck + s.s3_nch;
  S3Base* bS = s.s3_base;
  S3Base* bM = s.s3_base + s.s3_nch;
  const uint8_t* atS = s.s3_attr;
  const uint8_t* atM = s.s3_attr + s.s3_np;
  const int64_t m = c->mvict;
  const uint32_t cap = (uint32_t)s.s3_freq_cap, mm = (uint32_t)s.s3_move_min;
  if (threadIdx.x < kS3Bins) { hmain[threadIdx.x] = 0; hmov[threadIdx.x] = 0; }
  if (threadIdx.x < 8) sv[threadIdx.x] = -1;
  if (threadIdx.x == 0) {
    pl->lenS = lenS; pl->lenM = lenM;
    pl->ctr0 = c->s3_ctr;
    pl->hits = 0;
    pl->fb = 0;
  }
  __syncthreads();
  // ---- sizes: unpinned and victim-grade members of the small queue, main's unpinned
  const uint64_t tS = plan_scan(chS, [&](int64_t i) { return (uint64_t)ckS[i].nu << 32 | ckS[i].nev; },
                                [&](int64_t i, uint64_t ex, uint64_t) { bS[i].u = (uint32_t)(ex >> 32); bS[i].ev = (uint32_t)ex; });
  const int64_t K = (int64_t)(tS >> 32), T = (int64_t)(uint32_t)tS;
  const int64_t nS0 = (int64_t)plan_scan(chS, [&](int64_t i) { return (uint64_t)ckS[i].nlive; }, [&](int64_t, uint64_t, uint64_t) {});
  const int64_t UMo = (int64_t)plan_scan(chM, [&](int64_t i) { return (uint64_t)ckM[i].nu; },
                                         [&](int64_t i, uint64_t ex, uint64_t) { bM[i].u = (uint32_t)ex; });
  for (int64_t i = threadIdx.x; i < chM; i += kPT)
    for (int r = 0; r < kS3Bins; ++r)
      if (ckM[i].hist[r]) atomicAdd(&hmain[r], ckM[i].hist[r]);
  // ---- small phase: how many evictions take the small queue, and where they stop
  const int64_t D = nS0 - s.s3_small_cap;
  int64_t nA = 0;
  if (D >= 0 && K >= 1 && m > 0) {
    const int64_t Dp = tmin<int64_t>(D, K - 1);
    int64_t TD = 0;
    if (Dp >= 1) {
      // the chunk holding unpinned member number Dp, then the victims among the first Dp
      if (threadIdx.x == 0) { sv[0] = -1; sv[1] = -1; }
      plan_scan(chS, [&](int64_t i) { return (uint64_t)ckS[i].nu; }, [&](int64_t i, uint64_t ex, uint64_t v) {
        if ((int64_t)ex < Dp && Dp <= (int64_t)(ex + v)) sv[0] = i;
      });
      const int64_t cd = sv[0];
      if (cd < 0) { lost_locate(s); return; }
      const int64_t want = Dp - bS[cd].u;
      const int n = (int)tmin<int64_t>(kS3Chunk, lenS - cd * kS3Chunk);
      const uint8_t* at = atS + cd * kS3Chunk;
      chunk_scan(n, [&](int j) {
        const uint32_t a = at[j];
        return (uint64_t)a_un(a) << 32 | (uint64_t)(a_un(a) && a_f(a) < mm);
      }, [&](int, uint64_t incl, uint64_t own) {
        if ((own >> 32) && (int64_t)(incl >> 32) == want) sv[1] = (int64_t)(uint32_t)incl;
      });
      if (sv[1] < 0) { lost_locate(s); return; }
      TD = bS[cd].ev + sv[1];
    }
    nA = tmin<int64_t>(m, 1 + TD);
  }
  int64_t pcut = 0, kS = 0;
  if (nA > 0 && nA <= T) {
    if (threadIdx.x == 0) { sv[2] = -1; sv[3] = -1; }
    plan_scan(chS, [&](int64_t i) { return (uint64_t)ckS[i].nev; }, [&](int64_t i, uint64_t ex, uint64_t v) {
      if ((int64_t)ex < nA && nA <= (int64_t)(ex + v)) sv[2] = i;
    });
    const int64_t ce = sv[2];
    if (ce < 0) { lost_locate(s); return; }
    const int64_t want = nA - bS[ce].ev;
    const int n = (int)tmin<int64_t>(kS3Chunk, lenS - ce * kS3Chunk);
    const uint8_t* at = atS + ce * kS3Chunk;
    chunk_scan(n, [&](int j) { const uint32_t a = at[j]; return (uint64_t)(a_un(a) && a_f(a) < mm); },
               [&](int j, uint64_t incl, uint64_t own) {
                 if (own && (int64_t)incl == want) sv[3] = j;
               });
    if (sv[3] < 0) { lost_locate(s); return; }
    pcut = ce * kS3Chunk + sv[3] + 1;
    kS = nA;
  } else if (nA > T) {
    pcut = lenS;
    kS = T;
  }
  // ---- moved members (unpinned, f >= threshold, before the cut): per chunk and by frequency
  const int64_t cfull = pcut / kS3Chunk;            // chunks wholly before the cut
  const int64_t cpart = pcut % kS3Chunk ? cfull : -1;  // the chunk the cut falls in
  __shared__ uint32_t part_u, part_h[kS3Bins];
  if (threadIdx.x == 0) part_u = 0;
  if (threadIdx.x < kS3Bins) part_h[threadIdx.x] = 0;
  __syncthreads();
  if (cpart >= 0) {
    const uint8_t* at = atS + cpart * kS3Chunk;
    for (int j = threadIdx.x; j < (int)(pcut - cpart * kS3Chunk); j += kPT) {
      const uint32_t a = at[j];
      if (a_un(a)) {
        atomicAdd(&part_u, 1u);
        atomicAdd(&part_h[a_f(a)], 1u);
      }
    }
  }
  __syncthreads();
  auto mv_of = [&](int64_t i, int lo) -> uint32_t {  // movers of small chunk i with f >= lo
    uint32_t n = 0;
    if (i < cfull) {
      for (int r = tmax<int>(lo, (int)mm); r < kS3Bins; ++r) n += ckS[i].hist[r];
    } else if (i == cpart) {
      for (int r = tmax<int>(lo, (int)mm); r < kS3Bins; ++r) n += part_h[r];
    }
    return n;
  };
  const int64_t MA = (int64_t)plan_scan(chS, [&](int64_t i) { return (uint64_t)mv_of(i, 0); },
                                        [&](int64_t i, uint64_t ex, uint64_t) { bS[i].mv = (uint32_t)ex; });
  for (int64_t i = threadIdx.x; i < chS; i += kPT) {
    if (i < cfull) {
      for (int r = (int)mm; r < kS3Bins; ++r)
        if (ckS[i].hist[r]) atomicAdd(&hmov[r], ckS[i].hist[r]);
    } else if (i == cpart) {
      for (int r = (int)mm; r < kS3Bins; ++r)
        if (part_h[r]) atomicAdd(&hmov[r], part_h[r]);
    }
  }
  __syncthreads();
  const int64_t nL = UMo + MA;
  const int64_t mB = m - kS;
  if (cap >= (uint32_t)kS3Bins || mB > nL || (s.flags & PS_FLAG_S3_SEQUENTIAL)) {  // sequential kernel
    if (threadIdx.x == 0) pl->fb = 1;
    return;
  }
  // ---- main phase: the final round Rs and the position P of its last visit
  int Rs = 0;
  int64_t P = -1, rge_P1 = 0, rgt_P1 = 0, base_R = 0, base_Rm1 = 0, cpP = -1;
  if (mB > 0) {
    int64_t cum = 0, k = 0;
    for (int r = 0; r < kS3Bins; ++r) {
      const int64_t h = (int64_t)hmain[r] + hmov[r];
      if (cum + h >= mB) { Rs = r; k = mB - cum; break; }
      cum += h;
    }
    // reinsertions of the complete rounds: round r reinserts every member with f > r
    for (int r = 0; r < Rs; ++r) {
      int64_t gt = 0;
      for (int q = r + 1; q < kS3Bins; ++q) gt += (int64_t)hmain[q] + hmov[q];
      if (r < Rs - 1) base_Rm1 += gt;
      base_R += gt;
    }
    // the k-th member with f == Rs, in list order (main chunks, then small chunks)
    if (threadIdx.x == 0) { sv[4] = -1; sv[6] = -1; }
    plan_scan(chM + chS, [&](int64_t i) -> uint64_t {
      return i < chM ? ckM[i].hist[Rs] : (Rs >= (int)mm ? mv_of(i - chM, Rs) - mv_of(i - chM, Rs + 1) : 0u);
    }, [&](int64_t i, uint64_t ex, uint64_t v) {
      if ((int64_t)ex < k && k <= (int64_t)(ex + v)) { sv[4] = i; sv[5] = (int64_t)ex; }
    });
    if (sv[4] < 0) { lost_locate(s); return; }
    const int64_t cp = sv[4], want = k - sv[5];
    const bool inM = cp < chM;
    const int64_t ci = inM ? cp : cp - chM;
    const int n = (int)tmin<int64_t>(kS3Chunk, (inM ? lenM : lenS) - ci * kS3Chunk);
    const uint8_t* at = (inM ? atM : atS) + ci * kS3Chunk;
    const int64_t jlim = inM ? n : pcut - ci * kS3Chunk;  // small: members before the cut only
    // packed: eq (bits 0-15), member (16-31), f >= Rs (32-47), f > Rs (48-63)
    chunk_scan(n, [&](int j) -> uint64_t {
      const uint32_t a = at[j];
      const bool mem = a_un(a) && (inM || (j < jlim && a_f(a) >= mm));
      if (!mem) return 0;
      const uint32_t f = a_f(a);
      return (uint64_t)(f == (uint32_t)Rs) | 1ull << 16 | (uint64_t)(f >= (uint32_t)Rs) << 32 |
             (uint64_t)(f > (uint32_t)Rs) << 48;
    }, [&](int, uint64_t incl, uint64_t own) {
      if ((own & 0xFFFF) && (int64_t)(incl & 0xFFFF) == want) {
        sv[6] = (int64_t)((incl >> 16) & 0xFFFF) - 1;  // members before it in the chunk
        sv[7] = (int64_t)(incl >> 32);                  // ge (16 bits) | gt (16 bits) up to it
      }
    });
    if (sv[6] < 0) { lost_locate(s); return; }
    const int64_t before = sv[6];
    P = inM ? (int64_t)bM[ci].u + before : UMo + (int64_t)bS[ci].mv + before;
    // within the chunk; the chunk's list-order bases are added below
    rge_P1 = sv[7] & 0xFFFF;
    rgt_P1 = (sv[7] >> 16) & 0xFFFF;
    cpP = cp;
  }
  // ---- list-order bases of f >= Rs and f > Rs (main chunks, then small chunks)
  const uint64_t tg = plan_scan(chM + chS, [&](int64_t i) -> uint64_t {
    uint32_t ge = 0, gt = 0;
    if (i < chM) {
      for (int r = Rs; r < kS3Bins; ++r) ge += ckM[i].hist[r];
      gt = ge - ckM[i].hist[Rs];
    } else {
      ge = mv_of(i - chM, Rs);
      gt = mv_of(i - chM, Rs + 1);
    }
    return (uint64_t)ge << 32 | gt;
  }, [&](int64_t i, uint64_t ex, uint64_t) {
    S3Base& b = i < chM ? bM[i] : bS[i - chM];
    b.ge = (uint32_t)(ex >> 32);
    b.gt = (uint32_t)ex;
  });
  if (mB > 0) {
    const S3Base& b = cpP < chM ? bM[cpP] : bS[cpP - chM];
    rge_P1 += b.ge;
    rgt_P1 += b.gt;
  }
  const int64_t GE = (int64_t)(tg >> 32);
  const int64_t nG1 = Rs >= 1 ? GE - rge_P1 : 0;
  const int64_t nUnvMov = Rs == 0 ? nL - tmax<int64_t>(P + 1, UMo) : 0;
  const int64_t nMid = nG1 + nUnvMov + rgt_P1;
  // ---- kept entries: small = live and not consumed; main = pinned, or unvisited
  const int64_t nKeepS = (int64_t)plan_scan(chS, [&](int64_t i) -> uint64_t {
    const uint32_t cons = i < cfull ? ckS[i].nu : (i == cpart ? part_u : 0u);
    return ckS[i].nlive - cons;
  }, [&](int64_t i, uint64_t ex, uint64_t) { bS[i].keep = (uint32_t)ex; });
  const int64_t nKeepM = (int64_t)plan_scan(chM, [&](int64_t i) -> uint64_t {
    int64_t unv = 0;
    if (Rs == 0) unv = tmin<int64_t>(tmax<int64_t>((int64_t)bM[i].u + ckM[i].nu - (P + 1), 0), ckM[i].nu);
    return (uint64_t)(ckM[i].nlive - ckM[i].nu + unv);
  }, [&](int64_t i, uint64_t ex, uint64_t) { bM[i].keep = (uint32_t)ex; });
  // ---- the ghost FIFO: pushes, trimming, room
  __shared__ uint64_t gq;
  const uint64_t tail = c->ghost_tail, head = c->ghost_head;
  const int64_t live_old = c->ghost_live;
  const int64_t X = live_old + kS - s.s3_ghost_cap;
  const int64_t Xo = tmin<int64_t>(tmax<int64_t>(X, 0), live_old);
  const int64_t born = tmax<int64_t>(X - live_old, 0);
  const int gc = ((int64_t)(head - tail) + kS > (int64_t)s.ghost_ring_cap ||
                  ((s.flags & PS_FLAG_S3_COMPACT_GHOST) && head > tail)) ? 1 : 0;
  const uint64_t a0 = tail & ~(uint64_t)(kS3Chunk - 1);
  const int64_t nrch = head > tail ? cdiv64((int64_t)(head - a0), kS3Chunk) : 0;
  if (threadIdx.x == 0) gq = tail;
  __syncthreads();
  if (gc) {
    plan_scan(nrch, [&](int64_t i) { return (uint64_t)s.s3_rck[i]; },
              [&](int64_t i, uint64_t ex, uint64_t) { s.s3_rbase[i] = (uint32_t)ex; });
  } else if (Xo > 0 && born == 0) {
    // the Xo-th live position of the window: its ring chunk, then its word and bit
    if (threadIdx.x == 0) sv[2] = -1;
    plan_scan(nrch, [&](int64_t i) { return (uint64_t)s.s3_rck[i]; }, [&](int64_t i, uint64_t ex, uint64_t v) {
      if ((int64_t)ex < Xo && Xo <= (int64_t)(ex + v)) { sv[2] = i; sv[3] = (int64_t)ex; }
    });
    if (sv[2] < 0) { lost_locate(s); return; }
    const int64_t rc = sv[2];
    const uint64_t p0 = a0 + (uint64_t)rc * kS3Chunk;
    const uint32_t* rbits = bits_of(s, c->ghost_rbuf);
    const uint64_t rmask = s.ghost_ring_cap - 1;
    if (threadIdx.x < 32) {
      // a warp: two words a lane, in order
      uint32_t w[2];
      for (int h = 0; h < 2; ++h) {
        const uint64_t pw = p0 + 32u * (2 * threadIdx.x + h);
        uint32_t x = rbits[(pw & rmask) >> 5];
        if (pw < tail) x = tail - pw >= 32 ? 0u : x & (~0u << (uint32_t)(tail - pw));
        if (pw + 32 > head) x = head <= pw ? 0u : x & (~0u >> (uint32_t)(pw + 32 - head));
        w[h] = x;
      }
      const uint32_t n = __popc(w[0]) + __popc(w[1]);
      const uint32_t incl = warp_incl_scan(n);
      const int64_t want = Xo - sv[3];
      const int64_t exl = (int64_t)(incl - n);
      if (exl < want && want <= (int64_t)incl) {
        int64_t left = want - exl;
        const int h = left <= __popc(w[0]) ? 0 : 1;
        if (h == 1) left -= __popc(w[0]);
        const int bit = (int)__fns(w[h], 0, (int)left);
        gq = p0 + 32u * (2 * threadIdx.x + h) + (uint64_t)bit + 1;
      }
    }
    __syncthreads();
  }
  if (threadIdx.x == 0) {
    pl->pcut = pcut; pl->kS = kS; pl->MA = MA; pl->UMo = UMo; pl->nL = nL;
    pl->P = P; pl->Rs = Rs; pl->rge_P1 = rge_P1; pl->rgt_P1 = rgt_P1;
    pl->base_R = base_R; pl->base_Rm1 = base_Rm1;
    pl->nG1 = nG1; pl->nUnvMov = nUnvMov; pl->nMid = nMid;
    pl->nKeepS = nKeepS; pl->nKeepM = nKeepM;
    pl->ctr_end = c->s3_ctr + MA + base_R + rgt_P1;
    pl->gc = gc; pl->rbuf = c->ghost_rbuf;
    pl->g_head = head; pl->g_tail = tail; pl->ra0 = a0; pl->nrch = nrch;
    pl->live_old = live_old; pl->X = X; pl->born = born;
    pl->gctr0 = c->ghost_ctr;
    uint64_t q;
    if (gc) {
      pl->pbase = (uint64_t)(live_old - Xo) - (uint64_t)born;
      q = 0;
    } else {
      pl->pbase = head;
      q = born > 0 ? head + (uint64_t)born : (Xo > 0 ? gq : tail);
    }
    pl->q = q;
    // the ghost after the pushes and their trimming (hits come off at insertion)
    c->ghost_ctr += (uint64_t)kS;
    c->ghost_live = live_old - Xo + (kS - born);
    c->ghost_tail = q;
    c->ghost_head = pl->pbase + (uint64_t)kS;
    if (gc) c->ghost_rbuf ^= 1;
  }
}

// ===========================================================================
// 3. The published loop, one eviction at a time, on the same arrays: used
//    when the closed form does not apply (the main queue runs empty within the
//    step, or frequencies reach kS3Bins).  Writes what the plan's kernels
//    write: victims, moved and reinserted blocks, the new arrays' kept and
//    re-sequenced parts, the ghost pushes, and the plan's totals.
__global__ void k_s3_fallback(DevState s) {
  s = with_args(s);
  Ctl* c = s.ctl;
  S3Plan* pl = s.s3_plan;
  if (threadIdx.x != 0 || blockIdx.x != 0) return;
  if (c->status != PS_OK || !pl->fb) return;
  const int buf = c->s3_buf;
  const uint32_t* S = q_region(s, buf, 0);
  const uint32_t* M = q_region(s, buf, 1);
  uint32_t* oS = q_region(s, buf ^ 1, 0);
  uint32_t* oM = q_region(s, buf ^ 1, 1);
  const int64_t lenS = pl->lenS, lenM = pl->lenM, N = s.N;
  const uint32_t step32 = (uint32_t)c->step;
  const uint32_t mm = (uint32_t)s.s3_move_min;
  uint32_t* um = reinterpret_cast<uint32_t*>(s.csk);  // the main queue's unpinned members: a ring of N
  uint32_t* pushes = push_list(s);                    // the step's small-queue victims, in order
  auto live = [&](uint32_t b) { return (s.blk_flags[b] & 1) != 0; };
  auto unpinned = [&](uint32_t b) { return live(b) && s.blk_pin[b] != step32; };
  int64_t uh = 0, ut = 0, ucount = 0;
  for (int64_t j = 0; j < lenM; ++j) {
    const uint32_t b = M[j];
    if (unpinned(b)) { um[ut] = b; ut = ut + 1 == N ? 0 : ut + 1; ++ucount; }
  }
  int64_t nS = 0, Krem = 0;
  for (int64_t j = 0; j < lenS; ++j) {
    const uint32_t b = S[j];
    nS += live(b);
    Krem += unpinned(b);
  }
  const uint64_t ctr0 = c->s3_ctr;
  uint64_t ctr = ctr0;
  int64_t ps = 0, kS = 0, moved = 0;
  const int64_t m = c->mvict;
  int64_t budget = 4 * (N + 1) * ((int64_t)s.s3_freq_cap + 2) + lenS + 16;
  bool bad = false;
  auto evict_main = [&]() {
    for (;;) {
      if (ucount == 0 || --budget < 0) { bad = true; return; }
      const uint32_t b = um[uh];
      uh = uh + 1 == N ? 0 : uh + 1;
      --ucount;
      const uint32_t f = eff_freq(s, b);
      if (f > 0) {
        s.blk_freq[b] = f - 1;
        s.blk_s3seq[b] = ++ctr;
        um[ut] = b;
        ut = ut + 1 == N ? 0 : ut + 1;
        ++ucount;
      } else {
        mark_victim(s, b);
        return;
      }
    }
  };
  for (int64_t v = 0; v < m && !bad; ++v) {
    const bool use_small = (nS >= s.s3_small_cap && Krem > 0) || ucount == 0;
    bool done = false;
    if (use_small) {
      while (Krem > 0 && !bad) {
        uint32_t b = kNone;
        while (ps < lenS) {
          const uint32_t x = S[ps++];
          if (unpinned(x)) { b = x; break; }
        }
        if (b == kNone || --budget < 0) { bad = true; break; }
        --Krem;
        --nS;
        if (eff_freq(s, b) >= mm) {  // to the main queue's head
          s.blk_flags[b] |= 2;
          s.blk_s3seq[b] = ++ctr;
          um[ut] = b;
          ut = ut + 1 == N ? 0 : ut + 1;
          ++ucount;
          ++moved;
        } else {                     // out, its key into the ghost
          mark_victim(s, b);
          pushes[kS++] = b;
          done = true;
          break;
        }
      }
    }
    if (!done && !bad) evict_main();
  }
  // the new arrays' kept and re-sequenced parts
  int64_t nKeepS = 0, nKeepM = 0, nMid = 0;
  for (int64_t j = 0; j < lenS; ++j) {
    const uint32_t b = S[j];
    if (live(b) && !(j < ps && unpinned(b))) oS[nKeepS++] = b;
  }
  for (int64_t j = 0; j < lenM; ++j) {
    const uint32_t b = M[j];
    const bool vic = (s.bm_victim[b >> 5] >> (b & 31)) & 1;
    if (live(b) && !vic && s.blk_s3seq[b] <= ctr0) oM[nKeepM++] = b;
  }
  for (int64_t i = 0; i < ucount; ++i) {
    const uint32_t b = um[(uh + i) % N];
    if (s.blk_s3seq[b] > ctr0) oM[nKeepM + nMid++] = b;
  }
  // the ghost: trim the oldest live entries, compact when the ring lacks room, push
  const uint64_t rcap = s.ghost_ring_cap, rmask = rcap - 1;
  int rb = c->ghost_rbuf;
  uint64_t tail = c->ghost_tail, head = c->ghost_head;
  const int64_t live_old = c->ghost_live;
  const int64_t X = live_old + kS - s.s3_ghost_cap;
  const int64_t Xo = tmin<int64_t>(tmax<int64_t>(X, 0), live_old);
  const int64_t born = tmax<int64_t>(X - live_old, 0);
  uint32_t* ring = ring_of(s, rb);
  uint32_t* bits = bits_of(s, rb);
  auto bit_at = [&](uint32_t* bw, uint64_t p) { return (bw[(p & rmask) >> 5] >> (p & 31)) & 1; };
  int64_t erased = 0;
  while (erased < Xo && tail < head) {
    if (bit_at(bits, tail)) {
      gh_erase(s, ring[tail & rmask]);
      bits[(tail & rmask) >> 5] &= ~(1u << (tail & 31));
      ++erased;
    }
    ++tail;
  }
  uint64_t pbase = head;
  if ((int64_t)(head - tail) + kS > (int64_t)rcap || ((s.flags & PS_FLAG_S3_COMPACT_GHOST) && head > tail)) {
    uint32_t* nring = ring_of(s, rb ^ 1);
    uint32_t* nbits = bits_of(s, rb ^ 1);
    uint64_t w = 0;
    for (uint64_t p = tail; p < head; ++p) {
      if (!bit_at(bits, p)) continue;
      const uint32_t slot = ring[p & rmask];
      nring[w] = slot;
      s.ghost_map[slot].blk = (uint32_t)w;
      nbits[w >> 5] |= 1u << (w & 31);
      ++w;
    }
    for (uint64_t p = tail & ~31ull; p < head; p += 32) bits[(p & rmask) >> 5] = 0;
    rb ^= 1;
    ring = nring;
    bits = nbits;
    tail = 0;
    head = w;
    pbase = head - (uint64_t)born;
  } else if (born > 0) {
    tail = head + (uint64_t)born;
  }
  for (int64_t t = born; t < kS; ++t) {
    const uint32_t b = pushes[t];
    const uint64_t p = pbase + (uint64_t)t;
    const uint32_t slot = gh_insert(s, s.blk_key[b], s.blk_group[b], (uint32_t)(p & rmask), c->ghost_ctr + (uint64_t)t + 1);
    if (slot == kNone) { bad = true; break; }
    ring[p & rmask] = slot;
    bits[(p & rmask) >> 5] |= 1u << (p & 31);
  }
  c->ghost_ctr += (uint64_t)kS;
  c->ghost_live = live_old - Xo + (kS - born);
  c->ghost_tail = tail;
  c->ghost_head = pbase + (uint64_t)kS;
  c->ghost_rbuf = rb;
  pl->kS = kS;
  pl->MA = moved;
  pl->nKeepS = nKeepS;
  pl->nKeepM = nKeepM;
  pl->nMid = nMid;
  pl->ctr_end = ctr;
  if (bad) c->internal_error = 1;
}

// ===========================================================================
// 4. The plan applied, chunk by chunk: victims (the small queue's listed in
//    eviction order for their ghost pushes), moves and main-queue visits
//    (frequency, sequence number), the new arrays' kept and re-sequenced
//    parts; ring chunks of the FIFO window are trimmed, or compacted into the
//    other ring.  The ring chunks with work come first, so that no CTA takes
//    both a trimming chunk and a small-queue chunk before the others start.
__global__ void __launch_bounds__(kCT) k_s3_apply(DevState s) {
  s = with_args(s);
  Ctl* c = s.ctl;
  const S3Plan* pl = s.s3_plan;
  if (c->status != PS_OK || pl->fb) return;
  const int buf = c->s3_buf;
  const int64_t lenS = pl->lenS, lenM = pl->lenM;
  const int64_t chS = cdiv64(lenS, kS3Chunk), chM = cdiv64(lenM, kS3Chunk);
  const int64_t pcut = pl->pcut, UMo = pl->UMo, P = pl->P, MA = pl->MA;
  const int Rs = pl->Rs;
  const uint32_t mm = (uint32_t)s.s3_move_min;
  const uint64_t ctr0 = pl->ctr0;
  const uint64_t rmask = s.ghost_ring_cap - 1;
  const int rb = pl->rbuf, gc = pl->gc;
  uint32_t* ringO = ring_of(s, rb);
  uint32_t* bitsO = bits_of(s, rb);
  uint32_t* ringN = ring_of(s, gc ? rb ^ 1 : rb);
  uint32_t* bitsN = bits_of(s, gc ? rb ^ 1 : rb);
  const int64_t Xo = tmin<int64_t>(tmax<int64_t>(pl->X, 0), pl->live_old);
  // ring chunks with work: every chunk of the window when compacting, else
  // those before the new start
  int64_t nrw = 0;
  if (gc) nrw = pl->nrch;
  else if (Xo > 0) nrw = tmin<int64_t>(pl->nrch, cdiv64((int64_t)(pl->q - pl->ra0), kS3Chunk));
  const int64_t units = nrw + chS + chM;
  uint32_t* pushes = push_list(s);
  uint32_t* oS = q_region(s, buf ^ 1, 0);
  uint32_t* oM = q_region(s, buf ^ 1, 1);
  for (int64_t u0 = blockIdx.x; u0 < units; u0 += gridDim.x) {
    if (u0 >= nrw) {
      const int64_t u = u0 - nrw;
      const int r = u < chS ? 0 : 1;
      const int64_t ci = r ? u - chS : u;
      const int64_t len = r ? lenM : lenS;
      const int64_t j0 = ci * kS3Chunk + (int64_t)threadIdx.x * kPer;
      const uint4* ip = reinterpret_cast<const uint4*>(q_region(s, buf, r) + j0);
      const uint4 w0 = ip[0], w1 = ip[1];
      const uint32_t id[kPer] = {w0.x, w0.y, w0.z, w0.w, w1.x, w1.y, w1.z, w1.w};
      const uint2 ap = *reinterpret_cast<const uint2*>(s.s3_attr + (size_t)r * s.s3_np + j0);
      uint32_t a[kPer];
#pragma unroll
      for (int k = 0; k < 4; ++k) {
        a[k] = (ap.x >> (8 * k)) & 0xFF;
        a[k + 4] = (ap.y >> (8 * k)) & 0xFF;
      }
      // packed per-entry indicators (12-bit fields):
      //   small: ev, mv, keep, ge, gt      main: u, live, -, ge, gt
      uint64_t vals[kPer];
      uint64_t run = 0;
#pragma unroll
      for (int k = 0; k < kPer; ++k) {
        const uint32_t x = j0 + k < len ? a[k] : 0u;
        const bool live = a_live(x), un = a_un(x);
        const uint32_t f = a_f(x);
        uint64_t v;
        if (r == 0) {
          const bool cons = un && j0 + k < pcut;
          const bool ev = cons && f < mm, mv = cons && f >= mm;
          v = (uint64_t)ev | (uint64_t)mv << 12 | (uint64_t)(live && !cons) << 24 |
              (uint64_t)(mv && f >= (uint32_t)Rs) << 36 | (uint64_t)(mv && f > (uint32_t)Rs) << 48;
        } else {
          v = (uint64_t)un | (uint64_t)live << 12 | (uint64_t)(un && f >= (uint32_t)Rs) << 36 |
              (uint64_t)(un && f > (uint32_t)Rs) << 48;
        }
        vals[k] = run;  // exclusive within the thread
        run += v;
      }
      uint64_t tot;
      const uint64_t tex = block_excl_scan<uint64_t>(run, &tot);
      const S3Base bb = (r == 0 ? s.s3_base : s.s3_base + s.s3_nch)[ci];
#pragma unroll
      for (int k = 0; k < kPer; ++k) {
        const int64_t j = j0 + k;
        if (j >= len) break;
        const uint32_t x = a[k], b = id[k];
        if (!a_live(x)) continue;
        const uint64_t ex = tex + vals[k];
        const int64_t f0 = (int64_t)(ex & 0xFFF), f1 = (int64_t)((ex >> 12) & 0xFFF), f2 = (int64_t)((ex >> 24) & 0xFFF);
        const int64_t rge = bb.ge + (int64_t)((ex >> 36) & 0xFFF), rgt = bb.gt + (int64_t)((ex >> 48) & 0xFFF);
        const bool un = a_un(x);
        const uint32_t f = a_f(x);
        int64_t L = -1;         // list index when the entry is on the main phase's list
        bool mover = false;
        if (r == 0) {
          const bool cons = un && j < pcut;
          if (!cons) {
            q_put(s, oS, (int64_t)bb.keep + f2, b);
            continue;
          }
          if (f < mm) {  // small-queue victim: its key enters the ghost (k_s3_push)
            mark_victim(s, b);
            pushes[(int64_t)bb.ev + f0] = b;
            continue;
          }
          const int64_t mr = (int64_t)bb.mv + f1;  // moved to the main queue's head
          s.blk_flags[b] = 3;
          s.blk_s3seq[b] = ctr0 + 1 + (uint64_t)mr;
          L = UMo + mr;
          mover = true;
        } else {
          if (!un) {  // pinned: stays in place
            const int64_t U = f0, Lv = f1;
            int64_t unv = 0;
            if (Rs == 0) unv = U - tmin<int64_t>(U, tmax<int64_t>(0, P + 1 - (int64_t)bb.u));
            q_put(s, oM, (int64_t)bb.keep + (Lv - U) + unv, b);
            continue;
          }
          L = (int64_t)bb.u + f0;
        }
        // the main phase's visits of list member L
        if (P >= 0 && ((int)f < Rs || ((int)f == Rs && L <= P))) {
          mark_victim(s, b);
        } else if (L <= P) {  // reinserted in the final round
          s.blk_freq[b] = f - (uint32_t)Rs - 1;
          s.blk_s3seq[b] = ctr0 + (uint64_t)(MA + pl->base_R + rgt) + 1;
          q_put(s, oM, pl->nKeepM + pl->nG1 + pl->nUnvMov + rgt, b);
        } else if (Rs >= 1) {  // last reinserted in the round before
          s.blk_freq[b] = f - (uint32_t)Rs;
          s.blk_s3seq[b] = ctr0 + (uint64_t)(MA + pl->base_Rm1 + rge) + 1;
          q_put(s, oM, pl->nKeepM + (rge - pl->rge_P1), b);
        } else if (mover) {  // moved, not visited
          q_put(s, oM, pl->nKeepM + (L - tmax<int64_t>(P + 1, UMo)), b);
        } else {  // not visited: stays in place
          const int64_t U = f0, Lv = f1;
          const int64_t unv = U - tmin<int64_t>(U, tmax<int64_t>(0, P + 1 - (int64_t)bb.u));
          q_put(s, oM, (int64_t)bb.keep + (Lv - U) + unv, b);
        }
      }
    } else {
      // a ring chunk of the window [g_tail, g_head)
      const int64_t k = u0;
      const uint64_t p0 = pl->ra0 + (uint64_t)k * kS3Chunk;
      const uint64_t tail = pl->g_tail, head = pl->g_head;
      if (!gc && p0 >= pl->q) continue;  // trimming only: nothing at or past the new start
      // thread t: 8 positions, byte (t % 4) of word (t / 4)
      const int wi = threadIdx.x >> 2, by = threadIdx.x & 3;
      const uint64_t pw = p0 + 32u * wi;
      uint32_t word = bitsO[(pw & rmask) >> 5];
      if (pw < tail) word = tail - pw >= 32 ? 0u : word & (~0u << (uint32_t)(tail - pw));
      if (pw + 32 > head) word = head <= pw ? 0u : word & (~0u >> (uint32_t)(pw + 32 - head));
      const uint32_t mine = (word >> (8 * by)) & 0xFFu;
      if (gc) {
        uint32_t tot;
        const uint32_t ex = block_excl_scan<uint32_t>((uint32_t)__popc(mine), &tot);
        int64_t rank = (int64_t)s.s3_rbase[k] + ex;
        for (uint32_t mb = mine; mb; mb &= mb - 1, ++rank) {
          const uint64_t p = pw + 8u * by + (uint64_t)(__ffs(mb) - 1);
          const uint32_t slot = ringO[p & rmask];
          if (rank < Xo) {
            gh_erase(s, slot);
          } else {
            const uint64_t d = (uint64_t)(rank - Xo);
            ringN[d & rmask] = slot;
            s.ghost_map[slot].blk = (uint32_t)(d & rmask);
            atomicOr(bitsN + ((d & rmask) >> 5), 1u << (d & 31));
          }
        }
        // only the window's bits: near a full ring the first and last chunks
        // share words, whose other bits belong to the other chunk
        if (by == 0 && word) atomicAnd(bitsO + ((pw & rmask) >> 5), ~word);
      } else {
        for (uint32_t mb = mine; mb; mb &= mb - 1) {
          const uint64_t p = pw + 8u * by + (uint64_t)(__ffs(mb) - 1);
          if (p >= pl->q) break;
          gh_erase(s, ringO[p & rmask]);
          atomicAnd(bitsO + ((p & rmask) >> 5), ~(1u << (p & 31)));
        }
      }
    }
    __syncthreads();
  }
}

// 5. The step's ghost pushes, one thread each: the key of small-queue victim t
//    (in eviction order) enters the map with ghost sequence number gctr0 + t + 1
//    at FIFO position pbase + t; pushes the trimming removes at once
//    (t < born) are never written.
__global__ void __launch_bounds__(kCT) k_s3_push(DevState s) {
  s = with_args(s);
  Ctl* c = s.ctl;
  const S3Plan* pl = s.s3_plan;
  if (c->status != PS_OK || pl->fb) return;
  const int64_t kS = pl->kS, born = pl->born;
  const uint64_t rmask = s.ghost_ring_cap - 1;
  uint32_t* ring = ring_of(s, c->ghost_rbuf);  // the step's ring (the other one after a compaction)
  uint32_t* bits = bits_of(s, c->ghost_rbuf);
  const uint32_t* pushes = push_list(s);
  for (int64_t t = born + blockIdx.x * (int64_t)kCT + threadIdx.x; t < kS; t += (int64_t)gridDim.x * kCT) {
    const uint32_t b = pushes[t];
    const uint64_t p = pl->pbase + (uint64_t)t;
    const uint32_t slot = gh_insert(s, s.blk_key[b], s.blk_group[b], (uint32_t)(p & rmask), pl->gctr0 + (uint64_t)t + 1);
    if (slot == kNone) {
      c->internal_error = 1;
    } else {
      ring[p & rmask] = slot;
      atomicOr(bits + ((p & rmask) >> 5), 1u << (p & 31));
    }
  }
}

// ===========================================================================
// 6. After the insertions: each new block (in rank order, the order of its
//    sequence number) looks its key up in the ghost; a hit leaves the ghost
//    and enters the main queue, any other block the small queue.
__global__ void __launch_bounds__(kCT) k_s3_ins(DevState s) {
  s = with_args(s);
  Ctl* c = s.ctl;
  S3Plan* pl = s.s3_plan;
  if (c->status != PS_OK) return;
  const int64_t n_ins = c->need < c->n_alloc ? c->need : c->n_alloc;
  const int64_t r = blockIdx.x * (int64_t)kCT + threadIdx.x;
  bool hit = false;
  if (r < n_ins) {
    const uint32_t b = (uint32_t)s.out.admitted_ids[r];
    const uint64_t key = s.blk_key[b];
    const uint32_t g = s.blk_group[b];
    const uint32_t slot = gh_find(s, key, g);
    if (slot != kNone) {
      const uint32_t ridx = s.ghost_map[slot].blk;
      gh_erase_known(s, slot, key, g);
      atomicAnd(bits_of(s, c->ghost_rbuf) + (ridx >> 5), ~(1u << (ridx & 31)));
      s.blk_flags[b] = 3;
      hit = true;
    }
    s.blk_s3seq[b] = pl->ctr_end + (uint64_t)r + 1;
    s.s3_hit[r] = hit ? 1 : 0;
  }
  const uint32_t nh = block_sum<uint32_t>(hit ? 1u : 0u);
  if (threadIdx.x == 0 && nh) {
    atomicAdd(s.s3_ick + (blockIdx.x * (int64_t)kCT) / kS3Chunk, nh);
    atomicAdd(reinterpret_cast<unsigned long long*>(&pl->hits), (unsigned long long)nh);
  }
}

// 7. The new blocks' places: the small queue's after its kept members, the
//    main queue's after its kept and re-sequenced members, both in rank order.
__global__ void __launch_bounds__(kCT) k_s3_place(DevState s) {
  s = with_args(s);
  Ctl* c = s.ctl;
  const S3Plan* pl = s.s3_plan;
  if (c->status != PS_OK) return;
  const int64_t n_ins = c->need < c->n_alloc ? c->need : c->n_alloc;
  const int64_t r0 = blockIdx.x * (int64_t)kS3Chunk;
  if (r0 >= n_ins) return;
  // ghost hits of the earlier chunks
  __shared__ uint32_t wsum[kCT / 32];
  uint32_t before = 0;
  for (int64_t q = threadIdx.x; q < (int64_t)blockIdx.x; q += kCT) before += s.s3_ick[q];
  before = warp_sum(before);
  if (lane_id() == 0) wsum[threadIdx.x >> 5] = before;
  __syncthreads();
  before = 0;
#pragma unroll
  for (int w = 0; w < kCT / 32; ++w) before += wsum[w];
  const int64_t j0 = r0 + (int64_t)threadIdx.x * kPer;
  uint32_t h[kPer], own = 0;
#pragma unroll
  for (int k = 0; k < kPer; ++k) {
    h[k] = j0 + k < n_ins ? s.s3_hit[j0 + k] : 0u;
    own += h[k];
  }
  uint32_t tot;
  uint32_t hb = block_excl_scan<uint32_t>(own, &tot) + before;
  const int buf = c->s3_buf;
  uint32_t* oS = q_region(s, buf ^ 1, 0);
  uint32_t* oM = q_region(s, buf ^ 1, 1);
#pragma unroll
  for (int k = 0; k < kPer; ++k) {
    const int64_t rr = j0 + k;
    if (rr >= n_ins) break;
    const uint32_t b = (uint32_t)s.out.admitted_ids[rr];
    if (h[k]) {
      q_put(s, oM, pl->nKeepM + pl->nMid + hb, b);
      ++hb;
    } else {
      q_put(s, oS, pl->nKeepS + (rr - (int64_t)hb), b);
    }
  }
}

int32_t launch_s3_select(const DevState& s, cudaStream_t st, bool plain_first, int* launches) {
  if (plain_first) k_s3_count<<<152 * 4, kCT, 0, st>>>(s);
  else launch_k(k_s3_count, 152 * 4, kCT, 0, st, s);
  launch_k(k_s3_plan, 1, kPT, 0, st, s);
  launch_k(k_s3_fallback, 1, 32, 0, st, s);
  launch_k(k_s3_apply, 152 * 4, kCT, 0, st, s);
  launch_k(k_s3_push, 152 * 4, kCT, 0, st, s);
  *launches += 5;
  return cudaGetLastError() == cudaSuccess ? PS_OK : PS_ERR_CUDA;
}

int32_t launch_s3_insert(const DevState& s, cudaStream_t st, int* launches) {
  const int64_t B = s.max_blocks > 0 ? s.max_blocks : 1;
  launch_k(k_s3_ins, (int)((B + kCT - 1) / kCT), kCT, 0, st, s);
  launch_k(k_s3_place, (int)((B + kS3Chunk - 1) / kS3Chunk), kCT, 0, st, s);
  *launches += 2;
  return cudaGetLastError() == cudaSuccess ? PS_OK : PS_ERR_CUDA;
}

}  // namespace ps
