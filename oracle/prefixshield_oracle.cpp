// PrefixShield batched prefix-cache step: CPU ORACLE.
//
// TEST INFRASTRUCTURE ONLY.  This file is the plain, slow, single-threaded
// statement of what one step of the prefix cache computes.  It exists so that
// the CUDA library can be checked against it bit for bit.  Only the test
// suite, the smoke check and the CPU-baseline leg of the benchmark may load
// it.  It shares no code, header, table or constant generator with the CUDA
// library; everything here is written from the paper (Wang and Buyya,
// "Preserving Admission Responsibility in Multi-Tenant LLM Prefix Caches")
// and from the published definitions of SplitMix64, NH and S3-FIFO.
//
// Structure of one step (each stage cites the passage it follows):
//   S0 lazy token-bucket refill            Eq. 1 (evaluated at the step's clock)
//   S1 chained full-block hashing          Sec. III (native content-hash key)
//   S2 longest cached prefix lookup        Alg. 1 (n_cached), Sec. II-C namespaces
//   S3 grant of new blocks against the pool  (the batch reading of Alg. 1:
//                                          one Alg. 2 batch per step)
//   S4 per request, in request order:
//        OnRequest                          Alg. 1
//        OnTouch (debt-gated promotion)     Alg. 1, Eq. 4
//        OnCacheFullBlocks (metering)       Alg. 1, Eq. 2
//   S5 reclamation                         Alg. 2, Eq. 5-9 (prefixshield);
//                                          global recency (lru); S3-FIFO;
//                                          per-group recency inside equal
//                                          partitions (staticquota)
//   S6 eviction, id assignment, insertion
//
// Every function below is pinned by a CPU test (tests/test_oracle_*.py).
//
// Flag bits 4 and 8 (indexed queues, and their short first scan windows)
// select the CUDA library's victim data structure; the victims are the same,
// so this oracle ignores them.

#include <algorithm>
#include <cstdint>
#include <cstring>
#include <map>
#include <set>
#include <utility>
#include <vector>

namespace {

// ---- status codes (the oracle's own copy of the error vocabulary) ----------
constexpr int32_t OK = 0;
constexpr int32_t ERR_INVALID_ARG = -1;
constexpr int32_t ERR_CAPACITY = -2;
constexpr int32_t ERR_CLOCK = -3;

constexpr int32_t POLICY_LRU = 0;
constexpr int32_t POLICY_S3FIFO = 1;
constexpr int32_t POLICY_PREFIXSHIELD = 2;
constexpr int32_t POLICY_STATICQUOTA = 3;  // equal per-group partition, no borrowing (Sec. V-A)

// Retention classes, Sec. III-A: Probationary < Normal < Reuse (Eq. 9).
constexpr int32_t PROBATIONARY = 0;
constexpr int32_t NORMAL = 1;
constexpr int32_t REUSE = 2;

constexpr uint32_t FLAG_NO_SEGMENTATION = 1u;  // ablation: recency only (Sec. V-D)
constexpr uint32_t FLAG_NO_DEBT_GATE = 2u;     // ablation: promote regardless of debt

constexpr int MAX_CONTRACTS = 8;
constexpr int MAX_GROUPS = 1024;
constexpr int NUM_STATS = 15;
enum Stat {
  S_REQUESTS = 0, S_PROMPT_TOKENS, S_FULL_BLOCKS, S_HIT_BLOCKS, S_INSTEP_HIT_BLOCKS,
  S_HIT_TOKENS, S_ADMITTED_BLOCKS, S_UNGRANTED_BLOCKS, S_EVICTED_BLOCKS,
  S_INVALIDATED_BLOCKS, S_PROMOTIONS, S_GATED_REUSES, S_RESIDENT_BLOCKS,
  S_DEBT_RAW, S_DEBT_NORM
};

// Recency stamp (native free-queue order, Sec. III-D).  Every touch or
// admission of a step gets the next value of one running counter, in request
// order and, within a request, deepest block first: a request releases its
// blocks tail first, so its deeper blocks are older.  With `base` the number
// of full blocks of all earlier steps (plus one), request i's block m gets
//   base + (full blocks of requests 0..i-1) + (n_i - 1 - m).
// Limits: 2^18-1 requests per step and full blocks per request, 2^31-1 steps.
constexpr uint64_t MAX_POS = (1ull << 18) - 1;
constexpr uint64_t MAX_REQ = (1ull << 18) - 1;
constexpr uint64_t MAX_STEP = (1ull << 31) - 1;
uint64_t make_stamp(uint64_t base, uint64_t blocks_before, uint64_t n, uint64_t m) {
  return base + blocks_before + (n - 1 - m);
}

}  // namespace

extern "C" {

// The oracle's parameter block (field meaning: see include/prefixshield.h,
// which the oracle deliberately does not include).
typedef struct {
  int32_t num_contracts;
  int32_t fp_shift;
  int64_t epsilon_fp;
  int64_t rho_fp[MAX_CONTRACTS];
  int64_t beta_fp[MAX_CONTRACTS];
  int32_t contract_of_group[MAX_GROUPS];
  uint64_t hash_seed;
  int32_t s3_small_pct;
  int32_t s3_freq_cap;
  int32_t s3_move_min_freq;
  int32_t pad0;
  int64_t history_capacity;
  uint32_t flags;
  uint32_t pad1;
} orc_params_t;

typedef struct {
  int32_t* hit_blocks;        // [R]
  int32_t* admitted_blocks;   // [R]
  int32_t* admitted_offsets;  // [R+1]
  int32_t* admitted_ids;      // [cap]
  int32_t* evicted_ids;       // [cap]
  int32_t* invalidated_ids;   // [cap]
  int64_t* debt_raw;          // [G]
  int64_t* debt_norm;         // [G]
  int32_t n_admitted;
  int32_t n_evicted;
  int32_t n_invalidated;
  int32_t status;
} orc_out_t;

}  // extern "C"

namespace {

// ---------------------------------------------------------------------------
// SplitMix64 (Steele, Lea, Flood 2014; reference code by S. Vigna).
uint64_t splitmix64_next(uint64_t* state) {
  *state += 0x9E3779B97F4A7C15ull;
  uint64_t z = *state;
  z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
  z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
  return z ^ (z >> 31);
}
// The SplitMix64 output function alone, used as a 64-bit bijective mixer.
uint64_t mix64(uint64_t z) {
  z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
  z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
  return z ^ (z >> 31);
}

// NH (Black, Halevi, Krawczyk, Krovetz, Rogaway: UMAC, 1999): message words
// and key words are added mod 2^32 pairwise, the pair products taken as 64-bit
// values and summed mod 2^64.  'off' selects the Toeplitz-shifted key used
// for the second digest (UMAC's construction for a lower collision bound).
uint64_t nh_digest(const uint32_t* K, int off, const int32_t* M, int bs) {
  uint64_t sum = 0;
  for (int k = 0; k < bs / 2; ++k) {
    uint32_t a = (uint32_t)M[2 * k] + K[2 * k + off];
    uint32_t b = (uint32_t)M[2 * k + 1] + K[2 * k + 1 + off];
    sum += (uint64_t)a * (uint64_t)b;
  }
  return sum;
}

// Arithmetic modulo the Mersenne prime p = 2^61 - 1.
constexpr uint64_t P61 = (1ull << 61) - 1;
uint64_t mod61(uint64_t x) { return x % P61; }
uint64_t mulmod61(uint64_t a, uint64_t b) { return (uint64_t)(((unsigned __int128)a * b) % P61); }

// Chained content key of every full block of one token sequence (Sec. III,
// "native content-hash lookup key"; only full blocks are cached, Sec. III-B).
// Key schedule from SplitMix64(seed): bs+2 NH words, then the chain
// multiplier Kc and the digest multiplier Kd (both in [1, p)).
//   D_m = (NH0_m + Kd * NH2_m) mod p           (the block's 128-bit NH digest)
//   C_{-1} = mix(seed ^ (g+1)*phi) mod p       (namespace of group g)
//   C_m = (Kc * C_{m-1} + D_m) mod p           (chain over the prefix)
//   key_m = mix(C_m ^ (m+1)*c), with 0 and all-ones mapped to 1.
std::vector<uint64_t> chain_keys(uint64_t seed, int32_t group, int bs, const int32_t* tok, int64_t len) {
  std::vector<uint32_t> K(bs + 2);
  uint64_t st = seed;
  for (int j = 0; j < bs + 2; ++j) K[j] = (uint32_t)splitmix64_next(&st);
  uint64_t Kc = mod61(splitmix64_next(&st));
  uint64_t Kd = mod61(splitmix64_next(&st));
  if (Kc == 0) Kc = 1;
  if (Kd == 0) Kd = 1;
  int64_t n = len / bs;
  std::vector<uint64_t> keys(n);
  uint64_t C = mod61(mix64(seed ^ ((uint64_t)(group + 1) * 0x9E3779B97F4A7C15ull)));
  for (int64_t m = 0; m < n; ++m) {
    const int32_t* blk = tok + m * bs;
    uint64_t D = (mod61(nh_digest(K.data(), 0, blk, bs)) + mulmod61(Kd, mod61(nh_digest(K.data(), 2, blk, bs)))) % P61;
    C = (mulmod61(Kc, C) + D) % P61;
    uint64_t h = mix64(C ^ ((uint64_t)(m + 1) * 0xD1B54A32D192ED03ull));
    if (h == 0 || h == ~0ull) h = 1;
    keys[m] = h;
  }
  return keys;
}

// floor(a * b / c) for non-negative a, b and positive c, exact in 128 bits.
int64_t muldiv(int64_t a, int64_t b, int64_t c) {
  return (int64_t)(((__int128)a * (__int128)b) / (__int128)c);
}

struct Block {
  bool resident = false;
  uint64_t key = 0;
  int32_t group = 0;     // immutable accounting owner while resident (Sec. II-C)
  int32_t contract = 0;
  uint64_t prefix = 0;   // logical prefix id p (Sec. III-A)
  int32_t klass = 0;     // kappa(b) (Sec. III-A)
  uint64_t stamp = 0;    // native free-queue order (Sec. III-D)
  uint32_t acc = 0;      // access count (Sec. IV metadata)
  int32_t freq = 0;      // S3-FIFO frequency counter
  int32_t s3q = 0;       // S3-FIFO queue: 0 small, 1 main
  uint64_t s3seq = 0;    // S3-FIFO position (larger = nearer the head)
};

struct History {       // prefix-reference and admission history (Sec. IV)
  uint64_t refcount = 0;
  bool admitted = false;
};

// A block granted this step but not yet placed in the pool: its metadata is
// final before S6 chooses its id, so in-step touches update this record.
struct Pending {
  int32_t owner_req = 0;
  int32_t pos = 0;
  int32_t group = 0, contract = 0;
  uint64_t key = 0, prefix = 0;
  int32_t klass = 0;
  uint64_t stamp = 0;
  uint32_t acc = 0;
  int32_t freq = 0;
};

using GKey = std::pair<int32_t, uint64_t>;  // (group, key): namespace-scoped id

struct Oracle {
  int64_t N = 0;
  int32_t bs = 0, G = 0, policy = 0, C = 1;
  orc_params_t P{};
  std::vector<Block> blocks;
  std::map<GKey, int32_t> table;                 // native prefix table
  std::vector<int64_t> B;                        // B_{g,c}, fixed point
  int64_t t_prev = 0;                            // last refill time t0
  uint64_t step = 1;                             // index of the next step
  uint64_t stamp_base = 1;                       // first recency stamp of the next step
  std::map<GKey, History> history;               // keyed by (g, p)
  // S3-FIFO queues keyed by sequence number (head = largest).
  std::map<uint64_t, int32_t> s3_small, s3_main;
  uint64_t s3_ctr = 0;
  std::map<GKey, uint64_t> ghost;                // ghost entry -> sequence
  std::map<uint64_t, GKey> ghost_fifo;
  uint64_t ghost_ctr = 0;
  std::vector<int64_t> stats;                    // [G][NUM_STATS]
  int32_t sticky = OK;

  int64_t& stat(int g, int s) { return stats[(size_t)g * NUM_STATS + s]; }
  int64_t rho_min() const {
    int64_t r = P.rho_fp[0];
    for (int c = 1; c < C; ++c) r = std::min(r, P.rho_fp[c]);
    return r;
  }
  int32_t freq_cap() const { return P.s3_freq_cap; }
  int64_t s3_small_cap() const { return std::max<int64_t>(1, N * P.s3_small_pct / 100); }
  int64_t ghost_cap() const { return N - s3_small_cap(); }

  // Eq. 3: raw debt of group g from the stored balances.
  int64_t raw_debt(int g) const {
    int64_t d = 0;
    for (int c = 0; c < C; ++c) d += std::max<int64_t>(0, -B[(size_t)g * C + c]);
    return d;
  }
  // Eq. 5: normalized debt, w_c = rho_c / rho_min, each term floor-divided.
  int64_t norm_debt(int g) const {
    int64_t d = 0, rmin = rho_min();
    for (int c = 0; c < C; ++c) {
      int64_t def = std::max<int64_t>(0, -B[(size_t)g * C + c]);
      d += muldiv(def, rmin, P.rho_fp[c]);
    }
    return d;
  }
  // Eq. 8's decrement 1/W_g in fixed point, W_g = max weight of g's
  // currently indebted contracts; 0 when g has none.
  int64_t projected_decrement(int g) const {
    int64_t rmax = 0;
    for (int c = 0; c < C; ++c)
      if (B[(size_t)g * C + c] < 0) rmax = std::max(rmax, P.rho_fp[c]);
    if (rmax == 0) return 0;
    return muldiv((int64_t)1 << P.fp_shift, rho_min(), rmax);
  }
  // Order of candidates inside a group and in the global fallback (Eq. 9).
  std::pair<int32_t, uint64_t> order_key(const Block& b) const {
    int32_t k = (P.flags & FLAG_NO_SEGMENTATION) ? 0 : b.klass;
    return {k, b.stamp};
  }

  void remove_from_s3(int32_t id) {
    Block& b = blocks[id];
    if (b.s3q == 0) s3_small.erase(b.s3seq); else s3_main.erase(b.s3seq);
  }
  void ghost_push(const GKey& k) {
    uint64_t s = ++ghost_ctr;
    ghost[k] = s;
    ghost_fifo[s] = k;
    while ((int64_t)ghost.size() > ghost_cap()) {
      auto it = ghost_fifo.begin();
      ghost.erase(it->second);
      ghost_fifo.erase(it);
    }
  }
  void ghost_erase(const GKey& k) {
    auto it = ghost.find(k);
    ghost_fifo.erase(it->second);
    ghost.erase(it);
  }

  int32_t step_once(int64_t now, int32_t R, const int32_t* group, const int64_t* offsets,
                    const int32_t* tokens, const int32_t* contract_ids, const uint64_t* prefix_ids,
                    orc_out_t* out);
};

// ---------------------------------------------------------------------------
int32_t Oracle::step_once(int64_t now, int32_t R, const int32_t* group, const int64_t* offsets,
                          const int32_t* tokens, const int32_t* contract_ids,
                          const uint64_t* prefix_ids, orc_out_t* out) {
  // ---- input validation (state is left unchanged on any error) -----------
  if (sticky != OK) return sticky;
  if (now < t_prev) return ERR_CLOCK;
  if (R < 0 || (uint64_t)R > MAX_REQ) return ERR_INVALID_ARG;
  if (step > MAX_STEP) return ERR_CAPACITY;
  if (R > 0 && offsets[0] != 0) return ERR_INVALID_ARG;
  for (int32_t i = 0; i < R; ++i) {
    if (offsets[i + 1] < offsets[i]) return ERR_INVALID_ARG;
    if (group[i] < 0 || group[i] >= G) return ERR_INVALID_ARG;
    if (contract_ids && (contract_ids[i] < 0 || contract_ids[i] >= C)) return ERR_INVALID_ARG;
    if (prefix_ids && prefix_ids[i] == 0) return ERR_INVALID_ARG;
    if ((offsets[i + 1] - offsets[i]) / bs > (int64_t)MAX_POS) return ERR_INVALID_ARG;
  }

  // ---- S1: chained keys of every full block -------------------------------
  std::vector<std::vector<uint64_t>> keys(R);
  std::vector<int32_t> g(R), c(R);
  std::vector<uint64_t> p(R);
  std::vector<int64_t> n(R), before(R);  // before[i]: full blocks of requests 0..i-1
  for (int32_t i = 0; i < R; ++i) {
    g[i] = group[i];
    c[i] = contract_ids ? contract_ids[i] : P.contract_of_group[g[i]];
    keys[i] = chain_keys(P.hash_seed, g[i], bs, tokens + offsets[i], offsets[i + 1] - offsets[i]);
    n[i] = (int64_t)keys[i].size();
    before[i] = i ? before[i - 1] + n[i - 1] : 0;
    // The logical prefix id defaults to the key of the first full block.
    p[i] = prefix_ids ? prefix_ids[i] : (n[i] > 0 ? keys[i][0] : 0);
  }

  // History capacity: the number of live (g, p) entries after this step.
  {
    std::set<GKey> fresh;
    for (int32_t i = 0; i < R; ++i)
      if (n[i] > 0 && !history.count({g[i], p[i]})) fresh.insert({g[i], p[i]});
    if ((int64_t)(history.size() + fresh.size()) > P.history_capacity) {
      sticky = ERR_CAPACITY;
      return ERR_CAPACITY;
    }
  }

  // ---- S0: Eq. 1 lazy refill, evaluated at the step's clock for all (g,c).
  for (int gg = 0; gg < G; ++gg)
    for (int cc = 0; cc < C; ++cc) {
      int64_t& b = B[(size_t)gg * C + cc];
      int64_t beta = P.beta_fp[cc], rho = P.rho_fp[cc];
      int64_t need = beta - b;  // >= 0
      int64_t dt = now - t_prev;
      // min{beta, b + rho*dt} without overflow: dt >= ceil(need/rho) saturates.
      if (need <= 0 || dt >= (need + rho - 1) / rho) b = beta; else b += rho * dt;
    }
  t_prev = now;

  // ---- S2: longest cached prefix (n_cached of Alg. 1) ---------------------
  std::vector<int64_t> h(R, 0);
  std::set<int32_t> pinned;
  for (int32_t i = 0; i < R; ++i) {
    while (h[i] < n[i] && table.count({g[i], keys[i][h[i]]})) {
      pinned.insert(table[{g[i], keys[i][h[i]]}]);
      ++h[i];
    }
  }
  // Orphans: resident keys past a request's first miss cannot be reached by
  // lookup; they are dropped and re-materialized (reported as invalidated).
  std::set<int32_t> invalidated;
  for (int32_t i = 0; i < R; ++i)
    for (int64_t m = h[i] + 1; m < n[i]; ++m) {
      auto it = table.find({g[i], keys[i][m]});
      if (it != table.end() && !pinned.count(it->second)) invalidated.insert(it->second);
    }
  for (int32_t id : invalidated) {
    Block& b = blocks[id];
    table.erase({b.group, b.key});
    stat(b.group, S_INVALIDATED_BLOCKS) += 1;
    stat(b.group, S_RESIDENT_BLOCKS) -= 1;
    if (policy == POLICY_S3FIFO) remove_from_s3(id);
    b = Block{};
  }

  // Claims: each non-resident (g, key) belongs to the lowest request index
  // that contains it past its cached prefix (materialized once, charged once:
  // invariant I1).
  std::map<GKey, int32_t> owner;
  for (int32_t i = 0; i < R; ++i)
    for (int64_t m = h[i]; m < n[i]; ++m) {
      GKey k{g[i], keys[i][m]};
      if (!owner.count(k)) owner[k] = i;
    }
  std::vector<int64_t> s(R), cl(R);
  for (int32_t i = 0; i < R; ++i) {
    s[i] = n[i];
    for (int64_t m = h[i]; m < n[i]; ++m)
      if (owner[{g[i], keys[i][m]}] == i) { s[i] = m; break; }
    cl[i] = n[i] - s[i];
  }

  // ---- S3: grant new blocks against the pool ------------------------------
  // Claims are granted in (request, position) rank order while the pool
  // holds them: the whole pool (free + unpinned resident) for the shared
  // policies; for StaticQuota each group's own partition of Q = floor(N/G)
  // blocks minus its pinned blocks, ranked among its own requests.
  const int64_t quota = N / G;
  std::vector<int64_t> base(R), a(R), e(R), hit(R);
  if (policy == POLICY_STATICQUOTA) {
    std::vector<int64_t> pinned_g(G, 0), run_g(G, 0);
    for (int32_t id : pinned) pinned_g[blocks[id].group] += 1;
    for (int32_t i = 0; i < R; ++i) {
      base[i] = run_g[g[i]];
      run_g[g[i]] += cl[i];
      a[i] = std::min<int64_t>(cl[i], std::max<int64_t>(0, quota - pinned_g[g[i]] - base[i]));
    }
  } else {
    const int64_t avail = N - (int64_t)pinned.size();  // free + unpinned resident
    int64_t run = 0;
    for (int32_t i = 0; i < R; ++i) {
      base[i] = run;
      run += cl[i];
      a[i] = std::min<int64_t>(cl[i], std::max<int64_t>(0, avail - base[i]));
    }
  }
  // Request j's claims are ranked consecutively, so its key at position m is
  // granted iff it is among the first a_j of them.
  auto granted = [&](int32_t j, int64_t m) { return m - s[j] < a[j]; };
  for (int32_t i = 0; i < R; ++i) {
    e[i] = 0;
    for (int64_t m = h[i]; m < s[i]; ++m) {
      int32_t j = owner[{g[i], keys[i][m]}];
      if (granted(j, m)) ++e[i]; else break;
    }
    // When e_i < s_i - h_i some earlier claim is not granted, so neither is
    // any claim ranked after it in the same pool, and a_i is already 0: no
    // block is materialized past an ungranted one.
    hit[i] = h[i] + e[i];
  }

  // ---- S4: Alg. 1 hooks, request by request -------------------------------
  std::map<GKey, Pending> pending;
  const int64_t eps = P.epsilon_fp;
  const int64_t unit = (int64_t)1 << P.fp_shift;
  for (int32_t i = 0; i < R; ++i) {
    const int32_t gi = g[i];
    stat(gi, S_REQUESTS) += 1;
    stat(gi, S_PROMPT_TOKENS) += offsets[i + 1] - offsets[i];
    if (n[i] == 0) continue;  // no full block: no prefix id, no policy effect
    stat(gi, S_FULL_BLOCKS) += n[i];

    // OnRequest (Alg. 1): q_r = prior reference count, then record.
    History& hist = history[{gi, p[i]}];
    const uint64_t q = hist.refcount;
    hist.refcount += 1;
    const bool admitted_before = hist.admitted;

    // OnTouch (Alg. 1, Eq. 4) on the hit blocks H = cached prefix + in-step.
    const bool proven = (q >= 1) && admitted_before;
    const int64_t d = raw_debt(gi);  // D_g(t) before this request's charge
    const bool gate_open = (P.flags & FLAG_NO_DEBT_GATE) || d <= eps;
    for (int64_t m = 0; m < hit[i]; ++m) {
      const uint64_t st = make_stamp(stamp_base, (uint64_t)before[i], (uint64_t)n[i], (uint64_t)m);
      int32_t owner_g, owner_c, *klass;
      uint64_t owner_p, *stamp;
      uint32_t* acc;
      int32_t* freq;
      if (m < h[i]) {
        Block& b = blocks[table[{gi, keys[i][m]}]];
        owner_g = b.group; owner_c = b.contract; owner_p = b.prefix;
        klass = &b.klass; stamp = &b.stamp; acc = &b.acc; freq = &b.freq;
      } else {
        auto pit = pending.find({gi, keys[i][m]});
        if (pit == pending.end()) break;  // only reachable on a 64-bit key collision
        Pending& b = pit->second;
        owner_g = b.group; owner_c = b.contract; owner_p = b.prefix;
        klass = &b.klass; stamp = &b.stamp; acc = &b.acc; freq = &b.freq;
      }
      // UpdateAccessMetadata
      *stamp = std::max(*stamp, st);
      *acc += 1;
      *freq = std::min(freq_cap(), *freq + 1);
      // Promotion-eligible only for proven reuse of matching (g, c, p).
      if (proven && owner_g == gi && owner_c == c[i] && owner_p == p[i] && *klass != REUSE) {
        if (gate_open) {
          *klass = REUSE;
          stat(gi, S_PROMOTIONS) += 1;
        } else {
          stat(gi, S_GATED_REUSES) += 1;  // RecordDebtGatedReuse
        }
      }
    }
    stat(gi, S_HIT_BLOCKS) += hit[i];
    stat(gi, S_INSTEP_HIT_BLOCKS) += e[i];
    stat(gi, S_HIT_TOKENS) += hit[i] * bs;

    // OnCacheFullBlocks (Alg. 1): n_r = newly materialized full blocks.
    const int64_t nr = a[i];
    stat(gi, S_UNGRANTED_BLOCKS) += cl[i] - a[i];
    if (nr > 0) {
      int64_t& bal = B[(size_t)gi * C + c[i]];
      bal -= nr * unit;                                           // Eq. 2
      const int32_t k_new = (bal < -eps || !admitted_before) ? PROBATIONARY : NORMAL;
      hist.admitted = true;                                       // RecordSuccessfulAdmission
      stat(gi, S_ADMITTED_BLOCKS) += nr;
      for (int64_t m = s[i]; m < s[i] + nr; ++m) {                // AttachBlockMetadata
        Pending pb;
        pb.owner_req = i; pb.pos = (int32_t)m; pb.group = gi; pb.contract = c[i];
        pb.key = keys[i][m]; pb.prefix = p[i]; pb.klass = k_new;
        pb.stamp = make_stamp(stamp_base, (uint64_t)before[i], (uint64_t)n[i], (uint64_t)m);
        pending[{gi, keys[i][m]}] = pb;
      }
    }
  }

  // ---- S5: reclamation (Alg. 2 for prefixshield) -------------------------
  int64_t need = 0;
  for (int32_t i = 0; i < R; ++i) need += a[i];
  // StaticQuota: group g's new blocks first fill its partition's free part
  // (Q - resident_g); only the rest, m_g, evicts its own blocks.
  std::vector<int64_t> m_g(G, 0);
  int64_t quota_victims = 0;
  if (policy == POLICY_STATICQUOTA) {
    std::vector<int64_t> need_g(G, 0), res_g(G, 0);
    for (int32_t i = 0; i < R; ++i) need_g[g[i]] += a[i];
    for (int64_t id = 0; id < N; ++id)
      if (blocks[id].resident) res_g[blocks[id].group] += 1;
    for (int gg = 0; gg < G; ++gg) {
      m_g[gg] = std::max<int64_t>(0, need_g[gg] - (quota - res_g[gg]));
      quota_victims += m_g[gg];
    }
  }
  // TakeTrueFree: the smallest free ids first (work conservation, Sec. III-E).
  std::vector<int32_t> take;
  const int64_t want_free = need - quota_victims;
  for (int64_t id = 0; id < N && (int64_t)take.size() < want_free; ++id)
    if (!blocks[id].resident) take.push_back((int32_t)id);
  int64_t mvict = need - (int64_t)take.size();
  std::vector<int32_t> victims;
  if (mvict > 0) {
    if (policy == POLICY_STATICQUOTA) {
      // Each group reclaims its own m_g least recently released blocks.
      std::vector<std::set<std::pair<uint64_t, int32_t>>> q(G);
      for (int64_t id = 0; id < N; ++id)
        if (blocks[id].resident && !pinned.count((int32_t)id)) q[blocks[id].group].insert({blocks[id].stamp, (int32_t)id});
      for (int gg = 0; gg < G; ++gg) {
        auto it = q[gg].begin();
        for (int64_t v = 0; v < m_g[gg]; ++v, ++it) victims.push_back(it->second);
      }
    } else if (policy == POLICY_LRU) {
      // Global free-queue order: least recently released first.
      std::set<std::pair<uint64_t, int32_t>> q;
      for (int64_t id = 0; id < N; ++id)
        if (blocks[id].resident && !pinned.count((int32_t)id)) q.insert({blocks[id].stamp, (int32_t)id});
      auto it = q.begin();
      for (int64_t v = 0; v < mvict; ++v, ++it) victims.push_back(it->second);
    } else if (policy == POLICY_PREFIXSHIELD) {
      // SegmentQueuesByOwner + EffectiveDebtContext, then the Alg. 2 loop.
      using OK_ = std::pair<std::pair<int32_t, uint64_t>, int32_t>;
      std::vector<std::set<OK_>> Q(G);
      for (int64_t id = 0; id < N; ++id) {
        const Block& b = blocks[id];
        if (b.resident && !pinned.count((int32_t)id)) Q[b.group].insert({order_key(b), (int32_t)id});
      }
      std::vector<int64_t> Pg(G), delta(G);
      for (int gg = 0; gg < G; ++gg) { Pg[gg] = norm_debt(gg); delta[gg] = projected_decrement(gg); }
      for (int64_t v = 0; v < mvict; ++v) {
        int best = -1;
        for (int gg = 0; gg < G; ++gg) {
          if (Q[gg].empty() || Pg[gg] <= eps) continue;  // Eq. 6 membership
          if (best < 0 || Pg[gg] > Pg[best] ||
              (Pg[gg] == Pg[best] && Q[gg].begin()->first < Q[best].begin()->first))
            best = gg;                                     // Eq. 7 with its tie rule
        }
        int32_t id;
        if (best >= 0) {
          id = Q[best].begin()->second;                    // FirstSegmentQueue
          Q[best].erase(Q[best].begin());
          Pg[best] = std::max<int64_t>(0, Pg[best] - delta[best]);  // Eq. 8
        } else {
          int bg = -1;                                     // GlobalFirstSegmentQueue
          for (int gg = 0; gg < G; ++gg)
            if (!Q[gg].empty() && (bg < 0 || Q[gg].begin()->first < Q[bg].begin()->first)) bg = gg;
          id = Q[bg].begin()->second;
          Q[bg].erase(Q[bg].begin());
        }
        victims.push_back(id);
      }
    } else {
      // S3-FIFO (Yang et al., SOSP 2023), one eviction at a time.  Blocks hit
      // in this step are skipped in place: US / UM are the unpinned members
      // of the small and main queues, in queue order (tail = smallest seq).
      int64_t nS = (int64_t)s3_small.size();
      std::map<uint64_t, int32_t> US, UM;
      for (const auto& kv : s3_small) if (!pinned.count(kv.second)) US.insert(kv);
      for (const auto& kv : s3_main) if (!pinned.count(kv.second)) UM.insert(kv);
      auto evict_main = [&]() {
        for (;;) {
          auto it = UM.begin();
          int32_t id = it->second;
          Block& b = blocks[id];
          s3_main.erase(it->first);
          UM.erase(it);
          if (b.freq > 0) {           // reinsert at the head with one less
            b.freq -= 1;
            b.s3seq = ++s3_ctr;
            s3_main[b.s3seq] = id;
            UM[b.s3seq] = id;
          } else {
            victims.push_back(id);
            return;
          }
        }
      };
      for (int64_t v = 0; v < mvict; ++v) {
        bool use_small = (nS >= s3_small_cap() && !US.empty()) || UM.empty();
        if (!use_small) { evict_main(); continue; }
        bool done = false;
        while (!US.empty()) {
          auto it = US.begin();
          int32_t id = it->second;
          Block& b = blocks[id];
          s3_small.erase(it->first);
          US.erase(it);
          nS -= 1;
          if (b.freq >= P.s3_move_min_freq) {  // promote to the main queue head
            b.s3q = 1;
            b.s3seq = ++s3_ctr;
            s3_main[b.s3seq] = id;
            UM[b.s3seq] = id;
          } else {                             // evict into the ghost queue
            victims.push_back(id);
            ghost_push({b.group, b.key});
            done = true;
            break;
          }
        }
        if (!done) evict_main();
      }
    }
  }

  // ---- S6: evict, assign ids, insert --------------------------------------
  for (int32_t id : victims) {
    Block& b = blocks[id];
    table.erase({b.group, b.key});
    stat(b.group, S_EVICTED_BLOCKS) += 1;
    stat(b.group, S_RESIDENT_BLOCKS) -= 1;
    b = Block{};
  }
  std::vector<int32_t> alloc = take;
  alloc.insert(alloc.end(), victims.begin(), victims.end());
  std::sort(alloc.begin(), alloc.end());
  // Granted keys in (request, position) order receive ids in ascending order.
  int64_t r = 0;
  for (int32_t i = 0; i < R; ++i)
    for (int64_t m = s[i]; m < s[i] + a[i]; ++m) {
      const Pending& pb = pending.at({g[i], keys[i][m]});
      int32_t id = alloc[(size_t)r++];
      Block& b = blocks[id];
      b.resident = true;
      b.key = pb.key; b.group = pb.group; b.contract = pb.contract; b.prefix = pb.prefix;
      b.klass = pb.klass; b.stamp = pb.stamp; b.acc = pb.acc; b.freq = pb.freq;
      table[{b.group, b.key}] = id;
      stat(b.group, S_RESIDENT_BLOCKS) += 1;
      if (policy == POLICY_S3FIFO) {
        auto gh = ghost.find({b.group, b.key});
        if (gh != ghost.end()) { ghost_erase({b.group, b.key}); b.s3q = 1; }
        else b.s3q = 0;
        b.s3seq = ++s3_ctr;
        (b.s3q ? s3_main : s3_small)[b.s3seq] = id;
      }
    }

  // ---- outputs -----------------------------------------------------------
  std::sort(victims.begin(), victims.end());
  if (out) {
    int64_t off = 0;
    for (int32_t i = 0; i < R; ++i) {
      out->hit_blocks[i] = (int32_t)hit[i];
      out->admitted_blocks[i] = (int32_t)a[i];
      out->admitted_offsets[i] = (int32_t)off;
      off += a[i];
    }
    out->admitted_offsets[R] = (int32_t)off;
    for (size_t k = 0; k < alloc.size(); ++k) out->admitted_ids[k] = alloc[k];
    for (size_t k = 0; k < victims.size(); ++k) out->evicted_ids[k] = victims[k];
    size_t k = 0;
    for (int32_t id : invalidated) out->invalidated_ids[k++] = id;
    out->n_admitted = (int32_t)alloc.size();
    out->n_evicted = (int32_t)victims.size();
    out->n_invalidated = (int32_t)invalidated.size();
  }
  for (int gg = 0; gg < G; ++gg) {
    stat(gg, S_DEBT_RAW) = raw_debt(gg);
    stat(gg, S_DEBT_NORM) = norm_debt(gg);
    if (out) { out->debt_raw[gg] = raw_debt(gg); out->debt_norm[gg] = norm_debt(gg); }
  }
  if (out) out->status = OK;
  step += 1;
  stamp_base += R ? (uint64_t)(before[R - 1] + n[R - 1]) : 0;
  return OK;
}

}  // namespace

// ===========================================================================
// C ABI used by the Python test harness (oracle/__init__.py).
extern "C" {

int32_t orc_check_params(int64_t N, int32_t bs, int32_t G, int32_t policy, const orc_params_t* P) {
  if (!P || N <= 0 || N > (1ll << 30) || bs < 2 || bs > 256 || (bs & 1)) return ERR_INVALID_ARG;
  if (G <= 0 || G > MAX_GROUPS || policy < 0 || policy > 3) return ERR_INVALID_ARG;
  if (P->num_contracts < 1 || P->num_contracts > MAX_CONTRACTS) return ERR_INVALID_ARG;
  if (P->fp_shift < 0 || P->fp_shift > 30 || P->epsilon_fp < 0) return ERR_INVALID_ARG;
  int64_t rmin = P->rho_fp[0], rmax = P->rho_fp[0];
  for (int c = 0; c < P->num_contracts; ++c) {
    if (P->rho_fp[c] <= 0 || P->beta_fp[c] < 0) return ERR_INVALID_ARG;
    if (P->beta_fp[c] > (1ll << 52) || P->rho_fp[c] > (1ll << 52)) return ERR_INVALID_ARG;
    rmin = std::min(rmin, P->rho_fp[c]);
    rmax = std::max(rmax, P->rho_fp[c]);
  }
  // Eq. 8 decrement must be at least one fixed-point unit.
  if (muldiv((int64_t)1 << P->fp_shift, rmin, rmax) < 1) return ERR_INVALID_ARG;
  for (int gg = 0; gg < G; ++gg)
    if (P->contract_of_group[gg] < 0 || P->contract_of_group[gg] >= P->num_contracts) return ERR_INVALID_ARG;
  if (P->s3_small_pct < 1 || P->s3_small_pct > 100 || P->s3_freq_cap < 1 || P->s3_freq_cap > 255) return ERR_INVALID_ARG;
  if (P->s3_move_min_freq < 1 || P->history_capacity < 1) return ERR_INVALID_ARG;
  return OK;
}

void* orc_create(int64_t N, int32_t bs, int32_t G, int32_t policy, const orc_params_t* P) {
  if (orc_check_params(N, bs, G, policy, P) != OK) return nullptr;
  Oracle* o = new Oracle();
  o->N = N; o->bs = bs; o->G = G; o->policy = policy; o->P = *P; o->C = P->num_contracts;
  o->blocks.assign((size_t)N, Block{});
  o->B.assign((size_t)G * o->C, 0);
  for (int gg = 0; gg < G; ++gg)
    for (int c = 0; c < o->C; ++c) o->B[(size_t)gg * o->C + c] = P->beta_fp[c];  // B = beta at t = 0
  o->stats.assign((size_t)G * NUM_STATS, 0);
  return o;
}

void orc_destroy(void* h) { delete static_cast<Oracle*>(h); }

int32_t orc_step(void* h, int64_t now, int32_t R, const int32_t* group, const int64_t* offsets,
                 const int32_t* tokens, const int32_t* contract_ids, const uint64_t* prefix_ids,
                 orc_out_t* out) {
  if (!h) return ERR_INVALID_ARG;
  return static_cast<Oracle*>(h)->step_once(now, R, group, offsets, tokens, contract_ids, prefix_ids, out);
}

void orc_clear_status(void* h) { static_cast<Oracle*>(h)->sticky = OK; }

// Read-only: leading full blocks of each prompt resident now (n_cached of
// Alg. 1 against the current pool, no state change).
void orc_cached_prefix(void* h, int32_t R, const int32_t* group, const int64_t* offsets, const int32_t* tokens,
                       int32_t* out) {
  Oracle* o = static_cast<Oracle*>(h);
  for (int32_t i = 0; i < R; ++i) {
    std::vector<uint64_t> k = chain_keys(o->P.hash_seed, group[i], o->bs, tokens + offsets[i], offsets[i + 1] - offsets[i]);
    int32_t n = 0;
    while (n < (int32_t)k.size() && o->table.count({group[i], k[n]})) ++n;
    out[i] = n;
  }
}

void orc_stats(void* h, int64_t* out) {
  Oracle* o = static_cast<Oracle*>(h);
  std::memcpy(out, o->stats.data(), o->stats.size() * sizeof(int64_t));
}

// Per-block state, the ledger and the clock.  Arrays of length N / G*C.
void orc_export_blocks(void* h, uint8_t* resident, uint64_t* key, int32_t* group, int32_t* contract,
                       uint64_t* prefix, int32_t* klass, uint64_t* stamp, uint32_t* acc, int32_t* freq,
                       int32_t* s3q, uint64_t* s3seq) {
  Oracle* o = static_cast<Oracle*>(h);
  for (int64_t i = 0; i < o->N; ++i) {
    const Block& b = o->blocks[i];
    resident[i] = b.resident; key[i] = b.key; group[i] = b.group; contract[i] = b.contract;
    prefix[i] = b.prefix; klass[i] = b.klass; stamp[i] = b.stamp; acc[i] = b.acc;
    freq[i] = b.freq; s3q[i] = b.s3q; s3seq[i] = b.s3seq;
  }
}
void orc_export_ledger(void* h, int64_t* B, int64_t* t_prev, uint64_t* step, uint64_t* s3_ctr, uint64_t* ghost_ctr) {
  Oracle* o = static_cast<Oracle*>(h);
  std::memcpy(B, o->B.data(), o->B.size() * sizeof(int64_t));
  *t_prev = o->t_prev; *step = o->step; *s3_ctr = o->s3_ctr; *ghost_ctr = o->ghost_ctr;
}
// History entries sorted by (g, p); returns the count (arrays may be null to query).
int64_t orc_export_history(void* h, int32_t* g, uint64_t* p, uint64_t* refcount, uint8_t* admitted) {
  Oracle* o = static_cast<Oracle*>(h);
  int64_t k = 0;
  for (const auto& kv : o->history) {
    if (g) { g[k] = kv.first.first; p[k] = kv.first.second; refcount[k] = kv.second.refcount; admitted[k] = kv.second.admitted; }
    ++k;
  }
  return k;
}
// Ghost entries sorted by (g, key); returns the count.
int64_t orc_export_ghost(void* h, int32_t* g, uint64_t* key, uint64_t* seq) {
  Oracle* o = static_cast<Oracle*>(h);
  int64_t k = 0;
  for (const auto& kv : o->ghost) {
    if (g) { g[k] = kv.first.first; key[k] = kv.first.second; seq[k] = kv.second; }
    ++k;
  }
  return k;
}

// ---- building blocks exposed for the pin tests --------------------------
uint64_t orc_splitmix64_next(uint64_t* state) { return splitmix64_next(state); }
uint64_t orc_mix64(uint64_t z) { return mix64(z); }
uint64_t orc_nh(const uint32_t* K, int32_t off, const int32_t* M, int32_t bs) { return nh_digest(K, off, M, bs); }
int64_t orc_chain_keys(uint64_t seed, int32_t group, int32_t bs, const int32_t* tok, int64_t len, uint64_t* out) {
  std::vector<uint64_t> k = chain_keys(seed, group, bs, tok, len);
  for (size_t i = 0; i < k.size(); ++i) out[i] = k[i];
  return (int64_t)k.size();
}
uint64_t orc_make_stamp(uint64_t base, uint64_t blocks_before, uint64_t n, uint64_t m) {
  return make_stamp(base, blocks_before, n, m);
}

// The literal Alg. 2 victim loop on abstract inputs: G groups with projected
// scores P[g], decrements delta[g], and candidate keys per group (ascending,
// concatenated, qoff[g]..qoff[g+1]).  Writes the group and in-group index of
// each of the m victims in selection order.  Returns m.
int64_t orc_alg2_loop(int32_t G, const int64_t* P0, const int64_t* delta, int64_t eps, const int64_t* qoff,
                      const uint64_t* qkeys, int64_t m, int32_t* out_group, int64_t* out_index) {
  std::vector<int64_t> Pg(P0, P0 + G), head(G, 0);
  for (int64_t v = 0; v < m; ++v) {
    int best = -1;
    for (int gg = 0; gg < G; ++gg) {
      if (head[gg] >= qoff[gg + 1] - qoff[gg] || Pg[gg] <= eps) continue;
      if (best < 0 || Pg[gg] > Pg[best] ||
          (Pg[gg] == Pg[best] && qkeys[qoff[gg] + head[gg]] < qkeys[qoff[best] + head[best]]))
        best = gg;
    }
    if (best < 0) {
      for (int gg = 0; gg < G; ++gg)
        if (head[gg] < qoff[gg + 1] - qoff[gg] &&
            (best < 0 || qkeys[qoff[gg] + head[gg]] < qkeys[qoff[best] + head[best]]))
          best = gg;
      if (best < 0) return v;
    } else {
      Pg[best] = std::max<int64_t>(0, Pg[best] - delta[best]);
    }
    out_group[v] = best;
    out_index[v] = head[best]++;
  }
  return m;
}

}  // extern "C"
