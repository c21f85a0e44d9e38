// S3-FIFO baseline (Yang, Zhang, Qiu, Yue, Vinayak, SOSP 2023), the paper's
// reuse-aware replacement baseline (Sec. V-A): a small FIFO (10% of the
// pool), a main FIFO, a ghost FIFO of evicted small-queue keys, and a capped
// frequency counter, with no tenant metadata.
//
// Each eviction decides from the state the previous one left (which queue,
// whether the tail block moves or leaves), so the eviction batch of a step
// runs as one device thread over O(1) structures:
//   - each queue is a doubly linked list over block ids (tail = oldest);
//     blocks hit in the step are skipped in place by a per-step cursor;
//   - the ghost is a bucketed hash map (group, key) -> ring position plus a
//     FIFO ring of (key, group, sequence).
// Insertions run after the step's evictions, in rank order, also on one
// thread.  Every loop is bounded; a bound that is reached sets the step's
// internal-error flag instead of spinning.
#include "ps_internal.cuh"

namespace ps {

namespace {

__device__ __forceinline__ uint32_t eff_freq(const DevState& s, uint32_t b) {
  const uint32_t f = s.blk_freq[b];
  return f < (uint32_t)s.s3_freq_cap ? f : (uint32_t)s.s3_freq_cap;
}

struct Queues {
  uint32_t head[2], tail[2];
};

__device__ void q_unlink(const DevState& s, Queues& q, uint32_t b) {
  const uint32_t p = s.s3_prev[b], n = s.s3_next[b];
  if (p != kNone) s.s3_next[p] = n;
  else if (q.tail[0] == b) q.tail[0] = n;
  else q.tail[1] = n;
  if (n != kNone) s.s3_prev[n] = p;
  else if (q.head[0] == b) q.head[0] = p;
  else q.head[1] = p;
  s.s3_prev[b] = kNone;
  s.s3_next[b] = kNone;
}

__device__ void q_push_head(const DevState& s, Queues& q, int k, uint32_t b) {
  s.s3_prev[b] = q.head[k];
  s.s3_next[b] = kNone;
  if (q.head[k] != kNone) s.s3_next[q.head[k]] = b;
  else q.tail[k] = b;
  q.head[k] = b;
}

// ---- ghost: bucketed map (8 entries of {key, ring position, group}) -------
__device__ uint32_t ghost_home(const DevState& s, uint64_t key, uint32_t g) {
  return table_home(key, g, s.gh_nbuckets_log2);
}
__device__ uint32_t ghost_find(const DevState& s, uint64_t key, uint32_t g) {
  const uint32_t mask = (1u << s.gh_nbuckets_log2) - 1;
  uint32_t b = ghost_home(s, key, g);
  for (uint32_t it = 0; it <= mask; ++it) {
    // the bucket's ways and overflow count in one round of loads, then the
    // compares (a return among the loads would serialize them)
    TableEntry e[kTableWays];
#pragma unroll
    for (int w = 0; w < kTableWays; ++w) e[w] = s.ghost_map[(size_t)b * kTableWays + w];
    const uint32_t ovf = s.ghost_ovf[b];
    uint32_t hit = kNone;
#pragma unroll
    for (int w = kTableWays - 1; w >= 0; --w)
      if (e[w].blk != kNone && e[w].key == key && e[w].grp == g) hit = b * kTableWays + w;
    if (hit != kNone || ovf == 0) return hit;
    b = (b + 1) & mask;
  }
  return kNone;
}
__device__ bool ghost_insert(const DevState& s, uint64_t key, uint32_t g, uint32_t ring_pos) {
  const uint32_t mask = (1u << s.gh_nbuckets_log2) - 1;
  uint32_t b = ghost_home(s, key, g);
  for (uint32_t it = 0; it <= mask; ++it) {
    for (int w = 0; w < kTableWays; ++w) {
      TableEntry& e = s.ghost_map[(size_t)b * kTableWays + w];
      if (e.blk == kNone) {
        e.key = key;
        e.grp = g;
        e.blk = ring_pos;
        return true;
      }
    }
    s.ghost_ovf[b] += 1;
    b = (b + 1) & mask;
  }
  return false;
}
__device__ void ghost_erase(const DevState& s, uint32_t slot) {
  const uint32_t mask = (1u << s.gh_nbuckets_log2) - 1;
  TableEntry& e = s.ghost_map[slot];
  uint32_t x = ghost_home(s, e.key, e.grp);
  const uint32_t bucket = slot / kTableWays;
  for (uint32_t it = 0; x != bucket && it <= mask; ++it, x = (x + 1) & mask) s.ghost_ovf[x] -= 1;
  e.blk = kNone;
  e.key = 0;
  e.grp = 0;
}

// Ring position p holds a live entry iff the map points back at it.
__device__ bool ring_live(const DevState& s, uint64_t p) {
  const uint64_t rmask = s.ghost_ring_cap - 1;
  const uint32_t slot = ghost_find(s, s.ghost_ring_key[p & rmask], s.ghost_ring_grp[p & rmask]);
  return slot != kNone && s.ghost_map[slot].blk == (uint32_t)(p & rmask);
}

// Drop stale ring entries in place so a push has room (rarely needed).
__device__ void ring_compact(const DevState& s, Ctl* c) {
  const uint64_t rmask = s.ghost_ring_cap - 1;
  uint64_t w = c->ghost_tail;
  for (uint64_t p = c->ghost_tail; p < c->ghost_head; ++p) {
    if (!ring_live(s, p)) continue;
    if (w != p) {
      const uint32_t slot = ghost_find(s, s.ghost_ring_key[p & rmask], s.ghost_ring_grp[p & rmask]);
      s.ghost_ring_key[w & rmask] = s.ghost_ring_key[p & rmask];
      s.ghost_ring_grp[w & rmask] = s.ghost_ring_grp[p & rmask];
      s.ghost_ring_seq[w & rmask] = s.ghost_ring_seq[p & rmask];
      s.ghost_map[slot].blk = (uint32_t)(w & rmask);
    }
    ++w;
  }
  c->ghost_head = w;
}

// Evicted small-queue key enters the ghost; the oldest live entries leave
// while the ghost holds more than its capacity.
__device__ bool ghost_push(const DevState& s, Ctl* c, uint64_t key, uint32_t g) {
  const uint64_t rmask = s.ghost_ring_cap - 1;
  if (c->ghost_head - c->ghost_tail >= s.ghost_ring_cap) ring_compact(s, c);
  if (c->ghost_head - c->ghost_tail >= s.ghost_ring_cap) return false;
  const uint64_t p = c->ghost_head++;
  s.ghost_ring_key[p & rmask] = key;
  s.ghost_ring_grp[p & rmask] = g;
  s.ghost_ring_seq[p & rmask] = ++c->ghost_ctr;
  if (!ghost_insert(s, key, g, (uint32_t)(p & rmask))) return false;
  c->ghost_live += 1;
  while (c->ghost_live > s.s3_ghost_cap && c->ghost_tail < c->ghost_head) {
    const uint64_t t = c->ghost_tail++;
    if (!ring_live(s, t)) continue;
    ghost_erase(s, ghost_find(s, s.ghost_ring_key[t & rmask], s.ghost_ring_grp[t & rmask]));
    c->ghost_live -= 1;
  }
  return true;
}

}  // namespace

// Unlink the step's invalidated blocks, then choose the step's m victims.
__global__ void k_s3_evict(DevState s) {
  s = with_args(s);
  if (threadIdx.x != 0 || blockIdx.x != 0) return;
  Ctl* c = s.ctl;
  if (c->status != PS_OK) return;
  Queues q;
  for (int k = 0; k < 2; ++k) { q.head[k] = c->s3_head[k]; q.tail[k] = c->s3_tail[k]; }
  for (int64_t k = 0; k < c->s3_ninval; ++k) q_unlink(s, q, s.s3_inval[k]);
  const int64_t m = c->mvict;
  const uint32_t step32 = (uint32_t)c->step;
  int64_t nS = c->s3_nS, nM = c->s3_nM;
  int64_t uS = nS - c->s3_pinned[0], uM = nM - c->s3_pinned[1];
  uint32_t cur[2] = {q.tail[0], q.tail[1]};
  int64_t moved = 0;
  int64_t budget = 4 * (s.N + 1) * ((int64_t)s.s3_freq_cap + 2);  // bound on loop iterations
  bool bad = false;
  auto next_unpinned = [&](int k) -> uint32_t {
    while (cur[k] != kNone && s.blk_pin[cur[k]] == step32 && --budget > 0) cur[k] = s.s3_next[cur[k]];
    return cur[k];
  };
  auto evict = [&](uint32_t t) { s.bm_victim[t >> 5] |= 1u << (t & 31); };
  for (int64_t v = 0; v < m && !bad; ++v) {
    const bool use_small = (nS >= s.s3_small_cap && uS > 0) || uM == 0;
    bool done = false;
    if (use_small) {
      while (uS > 0 && budget-- > 0) {
        const uint32_t t = next_unpinned(0);
        if (t == kNone) { bad = true; break; }
        const uint32_t nxt = s.s3_next[t];
        q_unlink(s, q, t);
        cur[0] = nxt;
        nS -= 1;
        uS -= 1;
        if (eff_freq(s, t) >= (uint32_t)s.s3_move_min) {  // to the main queue's head
          s.blk_s3seq[t] = ++c->s3_ctr;
          s.blk_flags[t] |= 2;
          q_push_head(s, q, 1, t);
          if (cur[1] == kNone) cur[1] = t;
          nM += 1;
          uM += 1;
          moved += 1;
        } else {                                           // out, into the ghost
          evict(t);
          if (!ghost_push(s, c, s.blk_key[t], s.blk_group[t])) bad = true;
          done = true;
          break;
        }
      }
    }
    while (!done && !bad) {
      if (budget-- <= 0 || uM <= 0) { bad = true; break; }
      const uint32_t t = next_unpinned(1);
      if (t == kNone) { bad = true; break; }
      const uint32_t nxt = s.s3_next[t];
      q_unlink(s, q, t);
      const uint32_t f = eff_freq(s, t);
      if (f > 0) {  // reinsert at the head with one less
        s.blk_freq[t] = f - 1;
        s.blk_s3seq[t] = ++c->s3_ctr;
        q_push_head(s, q, 1, t);
        cur[1] = nxt == kNone ? t : nxt;
      } else {
        cur[1] = nxt;
        evict(t);
        nM -= 1;
        uM -= 1;
        done = true;
      }
    }
  }
  if (bad) c->internal_error = 1;
  for (int k = 0; k < 2; ++k) { c->s3_head[k] = q.head[k]; c->s3_tail[k] = q.tail[k]; }
  // victims leave the counts when they are dropped; moves are accounted here
  c->s3_nS -= moved;
  c->s3_nM += moved;
}

// Link the step's new blocks in rank order: a key found in the ghost enters
// the main queue (and leaves the ghost), any other the small queue.
__global__ void k_s3_insert(DevState s) {
  s = with_args(s);
  if (threadIdx.x != 0 || blockIdx.x != 0) return;
  Ctl* c = s.ctl;
  if (c->status != PS_OK) return;
  Queues q;
  for (int k = 0; k < 2; ++k) { q.head[k] = c->s3_head[k]; q.tail[k] = c->s3_tail[k]; }
  const int64_t need = c->need < c->n_alloc ? c->need : c->n_alloc;
  for (int64_t r = 0; r < need; ++r) {
    const uint32_t b = (uint32_t)s.out.admitted_ids[r];
    const uint32_t slot = ghost_find(s, s.blk_key[b], s.blk_group[b]);
    int k = 0;
    if (slot != kNone) {
      ghost_erase(s, slot);
      c->ghost_live -= 1;
      k = 1;
      s.blk_flags[b] |= 2;
    }
    s.blk_s3seq[b] = ++c->s3_ctr;
    q_push_head(s, q, k, b);
    if (k) c->s3_nM += 1; else c->s3_nS += 1;
  }
  for (int k = 0; k < 2; ++k) { c->s3_head[k] = q.head[k]; c->s3_tail[k] = q.tail[k]; }
}

void launch_s3_evict(const DevState& s, cudaStream_t st) { k_s3_evict<<<1, 32, 0, st>>>(s); }
void launch_s3_insert(const DevState& s, cudaStream_t st) { k_s3_insert<<<1, 32, 0, st>>>(s); }

}  // namespace ps
