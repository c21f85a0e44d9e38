// Indexed victim queues (PS_FLAG_INDEXED_QUEUES).
//
// The paper's selector scans every candidate and names indexed per-group,
// per-segment queues as the way to keep selection proportional to the
// victims (Sec. V-D overhead, Sec. VIII).  Here every queue is a log of
// (block, stamp) entries kept in stamp order:
//   * logs 3g + k: group g's blocks of retention class k (Eq. 9 segments);
//   * logs 3G + k: every group's blocks of class k (Alg. 2's global fallback
//     in (class, stamp) order, and lru over log 3G).
// Policies that ignore classes use k = 0 only; lru keeps only the global log,
// StaticQuota only the per-group logs.
//
// A block is appended to its logs at the end of every step that restamps it
// (a hit) or admits it; its older entries are left in place and become dead:
// an entry is live while its block is resident and still carries the entry's
// stamp (stamps are unique and only grow).  Every step's stamps exceed all
// earlier ones, and a step's appends go out in stamp order, so each log stays
// sorted by stamp and the oldest candidates of a log are its first live
// entries.  Per log the library keeps the number of live entries, which is
// the candidate count Alg. 2 and the quotas need, maintained as blocks are
// pinned, invalidated, taken and appended, so no step scans the pool.
//
// A select phase turns victim counts into "takes" (log, number of live
// entries to consume from its head) and scans a window past each head in
// 1024-entry chunks, one pass that counts, finds each chunk's place in its
// take by a decoupled look-back and marks; it repeats once over the rest of
// a log when dead entries made a window short.
// Logs live in one of two entry buffers; when a log lacks room for a step's
// appends, every log's live entries are compacted into the other buffer, in
// order, each log given room in proportion to its recent appends.
#include <climits>

#include "ps_device.cuh"
#include "ps_launch.cuh"

namespace ps {
namespace {

constexpr int kScanThreads = 256;          // 4 consecutive entries a thread per chunk
constexpr int kScanGrid = 152 * 8;         // grid-stride over the chunks of a scan
static_assert(kScanThreads * 4 == kLogChunk, "a scan CTA covers one chunk");

__device__ __forceinline__ const uint32_t* ent_blk(const DevState& s, int buf) { return s.lg_blk + (int64_t)buf * s.lg_P; }
__device__ __forceinline__ const uint64_t* ent_st(const DevState& s, int buf) { return s.lg_st + (int64_t)buf * s.lg_P; }

// Live: the block is resident and still carries the entry's stamp (and, in
// the fallback, was not taken by the debt phase).
__device__ __forceinline__ bool live_entry(const DevState& s, uint32_t b, uint64_t st, bool unvict) {
  if (b >= (uint64_t)s.N) return false;
  if (!(s.blk_flags[b] & 1) || s.blk_stamp[b] != st) return false;
  return !unvict || !((s.bm_victim[b >> 5] >> (b & 31)) & 1);
}

// The index t in [0, n) whose chunk range [c0[t], c0[t + 1]) holds chunk q.
__device__ __forceinline__ int range_of(const int32_t* c0, int n, int q) {
  int lo = 0, hi = n - 1;
  while (lo < hi) {
    const int mid = (lo + hi + 1) >> 1;
    if (c0[mid] <= q) lo = mid;
    else hi = mid - 1;
  }
  return lo;
}

// The block of stamp base + j, if that stamp is a block's current one (its
// last touch in this step, or its admission), and the logs it goes to.
__device__ __forceinline__ bool app_entry(const DevState& s, uint64_t base, int64_t j, int64_t nb, uint32_t* b,
                                          int32_t* A, int32_t* B) {
  *A = -1;
  *B = -1;
  if (j >= nb) return false;
  const uint32_t x = s.lg_slot[j];
  if (x >= (uint64_t)s.N || s.blk_stamp[x] != base + (uint64_t)j || !(s.blk_flags[x] & 1)) return false;
  const uint32_t g = s.blk_group[x], k = s.blk_klass[x];
  *A = lg_log_a(s, g, k);
  *B = lg_log_b(s, k);
  *b = x;
  return true;
}

// Last-CTA-done: true in the CTA that finishes last (after every CTA's writes).
__device__ __forceinline__ bool last_cta(Ctl* c) {
  __shared__ int s_last;
  __syncthreads();
  if (threadIdx.x == 0) {
    __threadfence();
    s_last = atomicAdd(&c->lg_ticket, 1u) == gridDim.x - 1;
  }
  __syncthreads();
  if (s_last) __threadfence();
  return s_last;
}

}  // namespace

__global__ void k_lg_init(DevState s) {
  const int64_t per = s.lg_P / s.lg_L;
  for (int l = threadIdx.x; l < s.lg_L; l += blockDim.x) {
    const int64_t a = per * l;
    s.lg_desc[l] = LogDesc{a, a, a, a + per};
    s.lg_live[l] = 0;
    s.lg_pin[l] = 0;
  }
}

// This step's pins leave their logs (the step has gone ahead); then the
// candidate counts Alg. 2 and the quotas read: |Q_g| and per class.
__global__ void __launch_bounds__(1024) k_lg_cand(DevState s) {
  s = with_args(s);
  Ctl* c = s.ctl;
  const bool ok = c->status == PS_OK;
  for (int l = threadIdx.x; l < s.lg_L; l += blockDim.x) {
    const int64_t p = s.lg_pin[l];
    if (p) {
      if (ok) s.lg_live[l] -= p;
      s.lg_pin[l] = 0;
    }
  }
  __syncthreads();
  if (!ok || s.policy == PS_LRU) return;
  for (int g = threadIdx.x; g < s.G; g += blockDim.x) {
    int64_t q = 0;
    for (int k = 0; k < kClasses; ++k) {
      const int64_t n = s.lg_live[g * kClasses + k];
      s.cls[g * kClasses + k].cnt = (uint32_t)n;
      q += n;
    }
    s.grp_qsize[g] = q;
  }
}

// The first scan round lists the phase's takes; every round sizes the window
// of each take still open (the first: a quarter more than the entries it
// still needs plus a chunk; the second: the rest of the log) and numbers the
// chunks.
__global__ void __launch_bounds__(1024) k_lg_plan(DevState s, int phase, int round) {
  s = with_args(s);
  Ctl* c = s.ctl;
  const bool ok = c->status == PS_OK;
  const bool more = round == 0 || c->lg_more;
  __syncthreads();
  if (threadIdx.x == 0) c->lg_more = 0;
  if (!ok || !more) {
    if (threadIdx.x == 0) {
      c->lg_nchunks = 0;
      if (round == 0) c->lg_ntk = 0;
    }
    return;
  }
  int ntk;
  if (round == 0) {
    const int64_t m = phase == 1 ? c->m_fb : c->mvict;
    const int nitems = (phase == 0 || phase == 3) ? s.G : 1;
    int base = 0;
    for (int i0 = 0; i0 < nitems; i0 += blockDim.x) {
      const int it = i0 + threadIdx.x;
      LogTake tk[kClasses];
      int nt = 0;
      if (m > 0 && it < nitems) {
        const bool per_group = phase == 0 || phase == 3;
        int64_t x = per_group ? s.grp_x[it] : m;
        const bool tie = phase == 0 && x > 0 && s.sel[it].incl == 2;
        const int ncls = (phase <= 1 && lg_segmented(s)) ? kClasses : 1;
        for (int k = 0; k < ncls && x > 0; ++k) {
          const int32_t l = per_group ? it * kClasses + k : s.G * kClasses + k;
          const int64_t w = tmin<int64_t>(x, s.lg_live[l]);
          x -= w;
          if (w > 0) {
            LogTake t{};
            t.want = w;
            t.log = l;
            t.tie = tie && x == 0;
            t.cur = s.lg_desc[l].head;
            tk[nt++] = t;
          }
        }
        if (x > 0) c->internal_error = 1;  // fewer candidates than the counts promised
      }
      int tot;
      const int ex = block_excl_scan(nt, &tot);
      for (int j = 0; j < nt; ++j) s.lg_tk[base + ex + j] = tk[j];
      base += tot;
    }
    ntk = base;
    if (threadIdx.x == 0) c->lg_ntk = ntk;
    __syncthreads();
  } else {
    ntk = c->lg_ntk;
  }
  int chunk_base = 0;
  for (int t0 = 0; t0 < ntk; t0 += blockDim.x) {
    const int t = t0 + threadIdx.x;
    int nch = 0;
    if (t < ntk) {
      LogTake k = s.lg_tk[t];
      if (!k.done) {
        if (round > 0) k.cur = k.wend;  // the last window held too few live entries
        const int64_t avail = s.lg_desc[k.log].tail - k.cur;
        const int64_t rem = k.want - k.got;
        const int64_t first = (s.flags & PS_FLAG_QUEUE_SHORT_WINDOWS) ? kLogChunk : rem + rem / 4 + kLogChunk;
        const int64_t wl = round == 0 ? tmin<int64_t>(avail, first) : avail;
        k.wend = k.cur + wl;
        nch = (int)((wl + kLogChunk - 1) / kLogChunk);
        if (nch == 0) c->internal_error = 1;  // victims owed by a log with nothing left to scan
        s.lg_tk[t] = k;
      }
    }
    int tot;
    const int ex = block_excl_scan(nch, &tot);
    if (t < ntk) s.lg_c0[t] = chunk_base + ex;
    chunk_base += tot;
  }
  if (threadIdx.x == 0) {
    s.lg_c0[ntk] = chunk_base;
    c->lg_nchunks = chunk_base;
    c->lg_ticket = 0;
  }
  for (int q = threadIdx.x; q < chunk_base; q += blockDim.x) s.lg_ck_out[q] = 0;  // k_lg_take's status words
}

// One take round in one pass (a decoupled look-back over the chunks of each
// take).  CTAs draw chunks in order from a ticket; each counts its chunk's
// live entries and publishes the count at once, then adds up the published
// counts of the take's earlier chunks (their inclusive prefix where already
// known) to learn how many of the take's live entries lie before it, and
// consumes the ones that fall within the take: victims marked in log order,
// live counts, the head.  A tied group's last entry is recorded for the tie
// rule instead.  The take's last chunk, if the window ended short, leaves
// the count for a second round.  Status words: 0 unpublished, kAgg | count,
// kIncl | inclusive prefix.  The wait for a predecessor is bounded.
constexpr uint64_t kAgg = 1ull << 62, kIncl = 2ull << 62, kValMask = (1ull << 62) - 1;
constexpr int kLookbackSpins = 1 << 22;

__global__ void __launch_bounds__(kScanThreads) k_lg_take(DevState s, int phase, cudaGraphConditionalHandle next,
                                                          int has_next) {
  s = with_args(s);
  __shared__ int32_t sc0[kMaxLogs + 1];
  __shared__ int s_q;
  __shared__ int64_t s_before;
  Ctl* c = s.ctl;
  const int nch = c->lg_nchunks;
  if (nch == 0) return;
  const int ntk = c->lg_ntk;
  for (int t = threadIdx.x; t <= ntk; t += blockDim.x) sc0[t] = s.lg_c0[t];
  const uint32_t* eb = ent_blk(s, c->lg_buf);
  const uint64_t* es = ent_st(s, c->lg_buf);
  unsigned long long* status = reinterpret_cast<unsigned long long*>(s.lg_ck_out);
  const int32_t gk = s.G * kClasses;
  for (;;) {
    __syncthreads();  // sc0 loaded; s_q, s_before of the last chunk consumed
    if (threadIdx.x == 0) s_q = (int)atomicAdd(&c->lg_ticket, 1u);
    __syncthreads();
    const int q = s_q;
    if (q >= nch) break;
    const int t = range_of(sc0, ntk, q);
    const LogTake k = s.lg_tk[t];
    const int qf = sc0[t], ql = sc0[t + 1] - 1;
    const int64_t e0 = k.cur + (int64_t)(q - qf) * kLogChunk + threadIdx.x * 4;
    uint32_t b[4];
    uint64_t st[4];
    bool live[4];
    int n = 0;
#pragma unroll
    for (int u = 0; u < 4; ++u) {
      const int64_t e = e0 + u;
      live[u] = false;
      if (e < k.wend) {
        b[u] = eb[e];
        st[u] = es[e];
        live[u] = live_entry(s, b[u], st[u], phase == 1);
      }
      n += live[u];
    }
    int tot;
    int64_t r = block_excl_scan(n, &tot);
    if (threadIdx.x == 0) {
      int64_t before = 0;
      if (q == qf) {
        atomicExch(status + q, kIncl | (uint64_t)tot);
      } else {
        atomicExch(status + q, kAgg | (uint64_t)tot);
        int j = q - 1, spins = 0;
        for (;;) {
          const uint64_t w = *reinterpret_cast<volatile unsigned long long*>(status + j);
          if (w & kIncl) {
            before += (int64_t)(w & kValMask);
            break;
          }
          if (w & kAgg) {
            before += (int64_t)(w & kValMask);
            --j;  // the take's first chunk publishes an inclusive prefix: j stays >= qf
            continue;
          }
          if (++spins > kLookbackSpins) {
            c->internal_error = 1;  // never expected: reported as a step status
            break;
          }
          __nanosleep(64);
        }
        atomicExch(status + q, kIncl | (uint64_t)(before + tot));
      }
      s_before = before;
    }
    __syncthreads();
    const int64_t rem = k.want - (k.got + s_before);  // the take's entries still to consume here
    int taken = 0;
    int32_t other[4];
#pragma unroll
    for (int u = 0; u < 4; ++u) {
      other[u] = -1;
      if (!live[u]) continue;
      if (r < rem) {
        const int64_t e = e0 + u;
        const bool last = r == rem - 1;
        if (last && k.tie) {
          const uint64_t key = lg_segmented(s) ? (st[u] | (uint64_t)s.blk_klass[b[u]] << 62) : st[u];
          s.lg_tie[k.log / kClasses] = TieItem{key, e, b[u], k.log};
          s.lg_desc[k.log].head = e;  // the tie candidate stays first in line
        } else {
          atomicOr(s.bm_victim + (b[u] >> 5), 1u << (b[u] & 31));
          ++taken;
          if (phase == 1) other[u] = lg_log_a(s, s.blk_group[b[u]], (uint32_t)(k.log - gk));
          if (last) s.lg_desc[k.log].head = e + 1;
        }
      }
      ++r;
    }
    // the debt phase's victims also leave their class's global log; the
    // fallback's leave their group's log
#pragma unroll
    for (int u = 0; u < 4; ++u) agg_add_i64(s.lg_live, (uint32_t)other[u], -1, other[u] >= 0);
    const int sum = block_sum(taken);
    if (threadIdx.x == 0) {
      if (sum) {
        atomic_add_i64(s.lg_live + k.log, -sum);
        if (phase == 0) {
          const int32_t B = lg_log_b(s, (uint32_t)(k.log % kClasses));
          if (B >= 0) atomic_add_i64(s.lg_live + B, -sum);
        }
        atomic_add_i64(&c->n_victims_marked, sum);
      }
      if (rem > 0 && rem <= tot) {
        s.lg_tk[t].done = 1;
      } else if (q == ql && rem > tot) {
        // the window ended short: every live entry in it is taken, and a
        // second round continues from its end
        s.lg_tk[t].got = k.got + s_before + tot;
        if (k.wend >= s.lg_desc[k.log].tail) {
          c->internal_error = 1;  // the log holds fewer live entries than counted
        } else {
          c->lg_more = 1;
          if (has_next) cudaGraphSetConditional(next, 1);
        }
      }
    }
  }
}

// Eq. 7's tie rule over the tied groups' recorded next candidates: the
// sel_k smallest (class, stamp) keys are taken.
__global__ void __launch_bounds__(1024) k_lg_tie(DevState s) {
  s = with_args(s);
  Ctl* c = s.ctl;
  if (c->status != PS_OK || c->mvict == 0 || c->sel_ntie == 0) return;
  __shared__ uint64_t skey[PS_MAX_GROUPS];
  __shared__ int16_t sgrp[PS_MAX_GROUPS];
  const int g = threadIdx.x;  // blockDim.x == PS_MAX_GROUPS
  const bool tied = g < s.G && s.sel[g].incl == 2 && s.grp_x[g] > 0;
  int n;
  const int ex = block_excl_scan((int)tied, &n);
  if (tied) {
    skey[ex] = s.lg_tie[g].key;
    sgrp[ex] = (int16_t)g;
  }
  __syncthreads();
  if (threadIdx.x == 0 && n != c->sel_ntie) c->internal_error = 1;
  const int k = c->sel_k;
  int taken = 0;
  if (threadIdx.x < n) {
    const uint64_t key = skey[threadIdx.x];
    int rank = 0;
    for (int j = 0; j < n; ++j) rank += skey[j] < key;
    const int gg = sgrp[threadIdx.x];
    if (rank < k) {
      const TieItem ti = s.lg_tie[gg];
      atomicOr(s.bm_victim + (ti.blk >> 5), 1u << (ti.blk & 31));
      atomic_add_i64(s.lg_live + ti.log, -1);
      const int32_t B = lg_log_b(s, (uint32_t)(ti.log % kClasses));
      if (B >= 0) atomic_add_i64(s.lg_live + B, -1);
      s.lg_desc[ti.log].head = ti.pos + 1;
      taken = 1;
    } else {
      s.grp_x[gg] -= 1;
    }
  }
  const int sum = block_sum(taken);
  if (threadIdx.x == 0 && sum) atomic_add_i64(&c->n_victims_marked, sum);
}

// ---- end of step: append this step's stamps, compacting first if needed ----

__global__ void __launch_bounds__(kAppChunk) k_lg_app_count(DevState s) {
  s = with_args(s);
  __shared__ uint32_t hist[kMaxLogs];
  Ctl* c = s.ctl;
  if (blockIdx.x == 0 && threadIdx.x == 0) {
    c->lg_cmp = 0;
    c->lg_ticket = 0;  // k_lg_take left its chunk count there
  }
  if (c->status != PS_OK) return;
  const int64_t nb = c->nblocks;
  const int q = blockIdx.x;
  if ((int64_t)q * kAppChunk >= nb) return;
  for (int l = threadIdx.x; l < s.lg_L; l += blockDim.x) hist[l] = 0;
  __syncthreads();
  uint32_t b;
  int32_t A, B;
  app_entry(s, c->stamp_base, (int64_t)q * kAppChunk + threadIdx.x, nb, &b, &A, &B);
  if (A >= 0) atomicAdd(&hist[A], 1u);
  if (B >= 0) atomicAdd(&hist[B], 1u);
  __syncthreads();
  for (int l = threadIdx.x; l < s.lg_L; l += blockDim.x) s.lg_app[(int64_t)l * s.lg_app_chunks + q] = hist[l];
}

// Per log (a CTA each): chunk offsets of the appends, their total, and
// whether the log has room for them.  Each thread scans a run of
// consecutive chunks, so the loads of a log's row are all in flight at once.
constexpr int kScanRun = 16;  // chunk counts a thread holds (up to 4096 x 16 chunks per pass)
__global__ void __launch_bounds__(256) k_lg_app_scan(DevState s, cudaGraphConditionalHandle hc, int has_cond) {
  s = with_args(s);
  Ctl* c = s.ctl;
  if (c->status != PS_OK) return;
  const int nch = (int)((c->nblocks + kAppChunk - 1) / kAppChunk);
  const int l = blockIdx.x;
  uint32_t* row = s.lg_app + (int64_t)l * s.lg_app_chunks;
  uint32_t before = 0;
  for (int base = 0; base < nch; base += (int)blockDim.x * kScanRun) {
    const int q0 = base + threadIdx.x * kScanRun;
    uint32_t v[kScanRun];
    uint32_t sum = 0;
#pragma unroll
    for (int u = 0; u < kScanRun; ++u) {
      v[u] = q0 + u < nch ? row[q0 + u] : 0u;
      sum += v[u];
    }
    uint32_t tot;
    uint32_t run = before + block_excl_scan(sum, &tot);
#pragma unroll
    for (int u = 0; u < kScanRun; ++u)
      if (q0 + u < nch) {
        row[q0 + u] = run;
        run += v[u];
      }
    before += tot;
  }
  if (threadIdx.x == 0) {
    s.lg_add[l] = before;
    const LogDesc d = s.lg_desc[l];
    if (d.tail + (int64_t)before > d.end) {
      c->lg_cmp = 1;
      if (has_cond) cudaGraphSetConditional(hc, 1);
    }
  }
}

// Compaction: chunks over every log's [head, tail).
__global__ void __launch_bounds__(1024) k_lg_cmp_plan(DevState s) {
  s = with_args(s);
  Ctl* c = s.ctl;
  if (c->status != PS_OK || !c->lg_cmp) {
    __syncthreads();
    if (threadIdx.x == 0) c->lg_nchunks = 0;
    return;
  }
  int base = 0;
  for (int l0 = 0; l0 < s.lg_L; l0 += blockDim.x) {
    const int l = l0 + threadIdx.x;
    int nch = 0;
    if (l < s.lg_L) {
      const LogDesc d = s.lg_desc[l];
      nch = (int)((d.tail - d.head + kLogChunk - 1) / kLogChunk);
    }
    int tot;
    const int ex = block_excl_scan(nch, &tot);
    if (l < s.lg_L) s.lg_c0[l] = base + ex;
    base += tot;
  }
  if (threadIdx.x == 0) {
    s.lg_c0[s.lg_L] = base;
    c->lg_nchunks = base;
  }
}

__global__ void __launch_bounds__(kScanThreads) k_lg_cmp_count(DevState s) {
  s = with_args(s);
  __shared__ int32_t sc0[kMaxLogs + 1];
  const Ctl* c = s.ctl;
  if (c->status != PS_OK || !c->lg_cmp) return;
  const int nch = c->lg_nchunks;
  if (nch == 0) return;
  const int L = s.lg_L;
  for (int t = threadIdx.x; t <= L; t += blockDim.x) sc0[t] = s.lg_c0[t];
  __syncthreads();
  const uint32_t* eb = ent_blk(s, c->lg_buf);
  const uint64_t* es = ent_st(s, c->lg_buf);
  for (int q = blockIdx.x; q < nch; q += gridDim.x) {
    const int l = range_of(sc0, L, q);
    const LogDesc d = s.lg_desc[l];
    const int64_t e0 = d.head + (int64_t)(q - sc0[l]) * kLogChunk + threadIdx.x * 4;
    int n = 0;
#pragma unroll
    for (int u = 0; u < 4; ++u) {
      const int64_t e = e0 + u;
      if (e < d.tail && live_entry(s, eb[e], es[e], false)) ++n;
    }
    const int tot = block_sum(n);
    if (threadIdx.x == 0) s.lg_ck[q] = (uint32_t)tot;
  }
}

// Per log (a CTA each): its live entries, and each chunk's offset inside it.
__global__ void __launch_bounds__(256) k_lg_cmp_live(DevState s) {
  s = with_args(s);
  Ctl* c = s.ctl;
  if (c->status != PS_OK || !c->lg_cmp) return;
  const int l = blockIdx.x;
  const int q0 = s.lg_c0[l], q1 = s.lg_c0[l + 1];
  int64_t before = 0;
  for (int base = q0; base < q1; base += (int)blockDim.x * kScanRun) {
    const int qa = base + threadIdx.x * kScanRun;
    uint32_t v[kScanRun];
    int64_t sum = 0;
#pragma unroll
    for (int u = 0; u < kScanRun; ++u) {
      v[u] = qa + u < q1 ? s.lg_ck[qa + u] : 0u;
      sum += v[u];
    }
    int64_t tot;
    int64_t run = before + block_excl_scan(sum, &tot);
#pragma unroll
    for (int u = 0; u < kScanRun; ++u)
      if (qa + u < q1) {
        s.lg_ck_out[qa + u] = run;
        run += v[u];
      }
    before += tot;
  }
  if (threadIdx.x == 0) {
    if (before != s.lg_live[l]) c->internal_error = 1;  // the live count drifted
    s.lg_new[l].tail = before;  // live count, for k_lg_cmp_layout
  }
}

// The new layout: each log gets its live entries, this step's appends, and a
// share of the free room in proportion to its appends (plus one).
__global__ void __launch_bounds__(1024) k_lg_cmp_layout(DevState s) {
  s = with_args(s);
  Ctl* c = s.ctl;
  if (c->status != PS_OK || !c->lg_cmp) return;
  const int L = s.lg_L;
  const int per = (L + (int)blockDim.x - 1) / (int)blockDim.x;
  const int l0 = threadIdx.x * per, l1 = l0 + per < L ? l0 + per : L;
  int64_t need = 0, wsum = 0;
  for (int l = l0; l < l1; ++l) {
    need += s.lg_new[l].tail + s.lg_add[l];
    wsum += s.lg_add[l] + 1;
  }
  const int64_t tot_need = block_sum(need), tot_w = block_sum(wsum);
  const int64_t room = s.lg_P - tot_need;
  if (room < 0 && threadIdx.x == 0) c->internal_error = 1;  // sized so that this cannot happen
  const int64_t free_room = room > 0 ? room : 0;
  int64_t caps = 0;
  for (int l = l0; l < l1; ++l) caps += s.lg_new[l].tail + s.lg_add[l] + free_room * (s.lg_add[l] + 1) / tot_w;
  int64_t tot_cap;
  int64_t start = block_excl_scan(caps, &tot_cap);
  for (int l = l0; l < l1; ++l) {
    const int64_t live = s.lg_new[l].tail;
    const int64_t cap = live + s.lg_add[l] + free_room * (s.lg_add[l] + 1) / tot_w;
    s.lg_new[l] = LogDesc{start, start, start + live, start + cap};
    start += cap;
  }
}

__global__ void __launch_bounds__(kScanThreads) k_lg_cmp_write(DevState s) {
  s = with_args(s);
  __shared__ int32_t sc0[kMaxLogs + 1];
  Ctl* c = s.ctl;
  if (c->status != PS_OK || !c->lg_cmp) return;
  const int nch = c->lg_nchunks;
  const int L = s.lg_L;
  for (int t = threadIdx.x; t <= L; t += blockDim.x) sc0[t] = s.lg_c0[t];
  __syncthreads();
  const int src = c->lg_buf;
  const uint32_t* eb = ent_blk(s, src);
  const uint64_t* es = ent_st(s, src);
  uint32_t* ob = s.lg_blk + (int64_t)(src ^ 1) * s.lg_P;
  uint64_t* os = s.lg_st + (int64_t)(src ^ 1) * s.lg_P;
  for (int q = blockIdx.x; q < nch; q += gridDim.x) {
    const int l = range_of(sc0, L, q);
    const LogDesc d = s.lg_desc[l];
    const int64_t e0 = d.head + (int64_t)(q - sc0[l]) * kLogChunk + threadIdx.x * 4;
    uint32_t b[4];
    uint64_t st[4];
    bool live[4];
    int n = 0;
#pragma unroll
    for (int u = 0; u < 4; ++u) {
      const int64_t e = e0 + u;
      live[u] = false;
      if (e < d.tail) {
        b[u] = eb[e];
        st[u] = es[e];
        live[u] = live_entry(s, b[u], st[u], false);
      }
      n += live[u];
    }
    int tot;
    int64_t o = s.lg_new[l].start + s.lg_ck_out[q] + block_excl_scan(n, &tot);
#pragma unroll
    for (int u = 0; u < 4; ++u)
      if (live[u]) {
        ob[o] = b[u];
        os[o] = st[u];
        ++o;
      }
  }
  if (last_cta(c)) {
    for (int l = threadIdx.x; l < L; l += blockDim.x) s.lg_desc[l] = s.lg_new[l];
    if (threadIdx.x == 0) {
      c->lg_buf = src ^ 1;
      c->lg_ticket = 0;
    }
  }
}

// Append in stamp order: within a chunk, entries of one log keep their
// order (warps take turns; lanes with the same log rank by lane).
__global__ void __launch_bounds__(kAppChunk) k_lg_app_write(DevState s) {
  s = with_args(s);
  __shared__ uint32_t cnt[kMaxLogs];
  Ctl* c = s.ctl;
  if (c->status != PS_OK) return;
  const int64_t nb = c->nblocks;
  const int q = blockIdx.x;
  const int L = s.lg_L;
  if ((int64_t)q * kAppChunk < nb) {
    for (int l = threadIdx.x; l < L; l += blockDim.x) cnt[l] = 0;
    __syncthreads();
    const int64_t j = (int64_t)q * kAppChunk + threadIdx.x;
    uint32_t b = 0;
    int32_t key[2];
    app_entry(s, c->stamp_base, j, nb, &b, &key[0], &key[1]);
    uint32_t rank[2] = {0, 0};
    const int w = threadIdx.x >> 5, lane = lane_id();
    const unsigned lt = (1u << lane) - 1;
    for (int turn = 0; turn < kAppChunk / 32; ++turn) {
      if (w == turn) {
#pragma unroll
        for (int i = 0; i < 2; ++i) {
          const unsigned peers = __match_any_sync(kFull, key[i]);
          const int leader = __ffs(peers) - 1;
          uint32_t base = 0;
          if (lane == leader && key[i] >= 0) {
            base = cnt[key[i]];
            cnt[key[i]] = base + (uint32_t)__popc(peers);
          }
          base = __shfl_sync(kFull, base, leader);
          rank[i] = base + (uint32_t)__popc(peers & lt);
        }
      }
      __syncthreads();
    }
    const int buf = c->lg_buf;
    uint32_t* ob = s.lg_blk + (int64_t)buf * s.lg_P;
    uint64_t* os = s.lg_st + (int64_t)buf * s.lg_P;
#pragma unroll
    for (int i = 0; i < 2; ++i)
      if (key[i] >= 0) {
        const int64_t o = s.lg_desc[key[i]].tail + s.lg_app[(int64_t)key[i] * s.lg_app_chunks + q] + rank[i];
        ob[o] = b;
        os[o] = c->stamp_base + (uint64_t)j;
      }
  }
  if (last_cta(c)) {
    for (int l = threadIdx.x; l < L; l += blockDim.x) {
      const int64_t a = s.lg_add[l];
      s.lg_desc[l].tail += a;
      s.lg_live[l] += a;
    }
    if (threadIdx.x == 0) c->lg_ticket = 0;
  }
}

// ---- host launchers -----------------------------------------------------------

void launch_queue_init(const DevState& s, cudaStream_t st) {
  if (s.lg_on) k_lg_init<<<1, 1024, 0, st>>>(s);
}

int32_t launch_queue_cand(const DevState& s, cudaStream_t st, int* launches) {
  k_lg_cand<<<1, 1024, 0, st>>>(s);  // may start a side branch: a plain launch
  ++*launches;
  return PS_OK;
}

int32_t launch_queue_select(const DevState& s, cudaStream_t st, const CaptureCtx* cap, int phase, int depth,
                            bool plain_first, int* launches) {
  cudaGraphConditionalHandle h1 = 0;
  if (cap && !cond_handle(st, &h1)) return PS_ERR_CUDA;
  auto round = [&](cudaStream_t q, int r) {
    if (plain_first && r == 0) k_lg_plan<<<1, 1024, 0, q>>>(s, phase, r);  // its predecessor is a join
    else launch_k(k_lg_plan, 1, 1024, 0, q, s, phase, r);
    launch_k(k_lg_take, kScanGrid, kScanThreads, 0, q, s, phase, h1, (cap && r == 0) ? 1 : 0);
    *launches += 2;
  };
  round(st, 0);
  if (cap) {
    // the second round is a conditional body (depth 0 phases nest on aux,
    // the fallback's on aux2)
    cudaStream_t body = depth == 0 ? cap->aux : cap->aux2;
    if (!cond_open(st, body, h1)) return PS_ERR_CUDA;
    round(body, 1);
    if (!cond_close(body)) return PS_ERR_CUDA;
  } else {
    round(st, 1);
  }
  if (phase == 0) {
    launch_k(k_lg_tie, 1, PS_MAX_GROUPS, 0, st, s);
    ++*launches;
  }
  return PS_OK;
}

int32_t launch_queue_append(const DevState& s, cudaStream_t st, const CaptureCtx* cap, int* launches) {
  const int ach = (int)s.lg_app_chunks;
  cudaGraphConditionalHandle hc = 0;
  if (cap && !cond_handle(st, &hc)) return PS_ERR_CUDA;
  launch_k(k_lg_app_count, ach, kAppChunk, 0, st, s);
  launch_k(k_lg_app_scan, s.lg_L, 256, 0, st, s, hc, cap ? 1 : 0);
  *launches += 2;
  cudaStream_t b = st;
  if (cap) {
    if (!cond_open(st, cap->aux, hc)) return PS_ERR_CUDA;
    b = cap->aux;
  }
  launch_k(k_lg_cmp_plan, 1, 1024, 0, b, s);
  launch_k(k_lg_cmp_count, kScanGrid, kScanThreads, 0, b, s);
  launch_k(k_lg_cmp_live, s.lg_L, 256, 0, b, s);
  launch_k(k_lg_cmp_layout, 1, 1024, 0, b, s);
  launch_k(k_lg_cmp_write, kScanGrid, kScanThreads, 0, b, s);
  *launches += 5;
  if (cap && !cond_close(cap->aux)) return PS_ERR_CUDA;
  launch_k(k_lg_app_write, ach, kAppChunk, 0, st, s);
  ++*launches;
  return PS_OK;
}

}  // namespace ps
