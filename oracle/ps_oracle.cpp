// Oracle for the PackServe scheduler hot path: TEST INFRASTRUCTURE, not part of the product.
//
// Only the tests, __graft_entry__.smoke() and bench.py's CPU-baseline / reference arm load this
// library.  It shares no code, header, table or constant generator with the CUDA library: it is a
// plain, single-threaded restatement of the paper's Algorithm 1 applied to one request at a time
// in arrival order, with instance state updated after every decision (Section 4, "Metadata
// service": state tracked along request paths).
//
// Data structures: one std::unordered_set<uint64_t> of cached block hashes per instance (the
// paper's Section 7 prefix tree, flattened: a block hash covers its whole prefix, so "prefix
// cached" == "block hash present").  Hit length = a linear walk along the request's chain until
// the first hash that is not in the set (exact whether or not the set is prefix-closed).
//
// Arithmetic: IEEE fp32 in the fixed operation order written below, built with
// -ffp-contract=off (no fused multiply-add) so that x86-64 and aarch64 give identical bits.
// Integer -> float conversions round to nearest.
//
// Readings where the paper is silent (each also listed in the design notes):
//  * Eq. 6 with the configuration's coefficients: T_pf(N,C) =
//    ((((a0 + a1 N) + a2 (N C)) + a3 (N N)) + a4 C) + a5 (C C); a4, a5 are the Section 5.3
//    empirical C and C^2 terms.
//  * Capacity guard (Alg. 1 CapacityCandidates): b + qr + 1 <= B_max and S + L <= M_KV.
//  * Eq. 8 is tested as (W - W_min) <= eta * Z (no division); Z <= 0 keeps all of A.
//  * TPOT, configuration form: ((b0 + b1 B) + b2 S') f + g_q (q + n), B = b + qr + 1, S' = S + L,
//    f = EMA factor of B's decode-batch segment (Section 5.3).  Paper form (Eq. 9):
//    ((b0 + b1 B) + b2 S') f + [b + qr > 0] T_pf(n,c) / max(1, L_out).
//  * TTFT (Eq. 4): T_pf(n,c) + (a0 qr + a1 q), overhead neglected; the budget is
//    max(target, T_pf(L,0)) (Section 8.1 Metrics); TTFT uses <=, TPOT uses strict < (Alg. 1).
//  * Policy variants of the evaluation (Section 8.3; off by default): Table 3's admission
//    ablations switch the KVC-first filter (C = A when off) and the SLO admission (T = C when off;
//    the TTFT test goes with the TPOT test) and replace the LMetric fallback by the D-C-Q order
//    over C; Table 4's selectors order T by D, D-Q, D-C, D-Q-C or H-C-Q, H being the predicted TPOT
//    headroom target - TPOT (fp32), smallest first.  Every order ends with the lowest id.
//  * Packing key D-C-Q (Section 6.2, Table 4): more decoding b, then more cached blocks h, then
//    fewer queued requests qr, then the lowest instance id.  Fallback CacheAwareLB = LMetric
//    (Section 6, Section 8.1 Baselines): min over C of (q + n)(b + qr + 1), lowest id on ties.
//  * Streaming windows (the paper leaves engine progress to the serving engine; these are the
//    simulation rules of the streaming workload).  Each instance keeps a FIFO queue of admitted
//    requests (remaining uncached prefill tokens) and a set of decoding requests (remaining output
//    tokens).  Advancing one window of window_ms: (1) every decoding request emits
//    k = max(1, floor(window_ms / ((b0 + b1 b) + b2 S))) tokens (fp32, b and S at the window start),
//    S grows by the tokens emitted, and a request whose output is exhausted leaves (b -= 1,
//    S -= L + out); (2) the queue drains prefill_tokens tokens in FIFO order, a request whose prefill
//    completes starts decoding (qr -= 1, b += 1); (3) while the cache holds more than cap blocks, the
//    leaf block (no cached child) with the smallest (last_use, hash) is evicted.  Scheduling stamps
//    last_use = window id on every block of an admitted request's chain (cached prefix and new
//    blocks) on its instance.

#include <cstdint>
#include <cstring>
#include <vector>
#include <unordered_set>
#include <unordered_map>
#include <algorithm>
#include <deque>
#include <set>

extern "C" {

typedef struct {
  float a0, a1, a2, a3, a4, a5;    // Eq. 6 (+ Section 5.3 C, C^2 terms)
  float b0, b1, b2;                // Eq. 7
  float g_q;                       // TPOT per queued prefill token (configuration form)
  float eta;                       // recompute budget (Eq. 8)
  float lout_median;               // Eq. 9 amortisation length
  int32_t interference_mode;       // 0 configuration form, 1 paper Eq. 9 form
  int32_t ttft_filter;             // 1: TTFT test in the admission set, 0: Alg. 1 exactly
  int32_t nseg;                    // decode-batch segments of the EMA factor table
  int32_t seg_lo[16];              // segment s covers B >= seg_lo[s] (ascending)
  float ema_factor[16];
  // Policy variants of the evaluation's ablations (Section 8.3, Table 3 and Table 4); the defaults
  // (1, 1, 0, 0) are Algorithm 1 as above.
  int32_t cache_filter;            // 1: KVC-first filter (Eq. 8); 0: C = A
  int32_t slo_filter;              // 1: TPOT (and TTFT) admission; 0: T = C
  int32_t fallback;                // with T empty: 0 LMetric over C, 1 the D-C-Q order over C
  int32_t selector;                // order inside T: 0 D-C-Q, 1 D, 2 D-Q, 3 D-C, 4 D-Q-C, 5 H-C-Q
} orc_model;

typedef struct { int32_t b, qr; int64_t q, S, M_KV; int32_t B_max; } orc_inst;

}  // extern "C"

namespace {

struct BlockMeta { uint64_t parent; uint32_t children; uint32_t last_use; };

struct Oracle {
  uint32_t I;
  orc_model m;
  std::vector<std::unordered_set<uint64_t>> cache;
  std::vector<orc_inst> st;
  // Leaf-first LRU bookkeeping (streaming windows only): per instance, block -> metadata, and the
  // set of leaves ordered by (last_use, hash).
  bool track = false;
  std::vector<std::unordered_map<uint64_t, BlockMeta>> meta;
  std::vector<std::set<std::pair<uint32_t, uint64_t>>> leaves;
  // Requests in flight (streaming windows only).
  struct Queued { uint32_t L, out; uint64_t rem; };
  struct Decoding { uint32_t L, out, rem; };
  std::vector<std::deque<Queued>> queue;
  std::vector<std::vector<Decoding>> decoding;
  std::vector<uint64_t> cap;
};

// Eq. 6 in the fixed order above.
float t_pf(const orc_model& m, float N, float C) {
  float t = m.a0 + m.a1 * N;
  t = t + m.a2 * (N * C);
  t = t + m.a3 * (N * N);
  t = t + m.a4 * C;
  t = t + m.a5 * (C * C);
  return t;
}

// Hit length: cached prefix blocks of the chain on instance i (Section 7 prefix-tree lookup).
uint64_t hit_len(const Oracle& o, uint32_t i, const uint64_t* chain, uint64_t nb) {
  uint64_t h = 0;
  while (h < nb && o.cache[i].count(chain[h])) ++h;
  return h;
}

float ema_factor(const orc_model& m, int64_t B) {
  int s = 0;
  for (int k = 0; k < m.nseg; ++k)
    if ((int64_t)m.seg_lo[k] <= B) s = k;
  return m.ema_factor[s];
}

struct Row {
  std::vector<uint64_t> hit;
  std::vector<float> tpot, ttft;
  std::vector<uint8_t> cls;    // 0: in T, 1: in C \ T, 2: in A \ C, 3: not in A
  int32_t pick = -1;
  uint8_t path = 2;            // 0 packed (from T), 1 fallback (LMetric over C), 2 reject
  bool anyA = false;           // A is not empty (over this oracle's instances)
  float Wmin = 0.f;            // min of W over A (over this oracle's instances), when anyA
};

// A W_min that replaces the one over this oracle's own instances: the oracle then holds one column
// block of a larger instance pool, and W_min is the minimum over the whole pool's A (Algorithm 1
// takes W_min over every capacity-eligible instance).
struct WminOverride { bool given = false; float Wmin = 0.f; };

// Algorithm 1 for one request against the current caches and state.
void decide(const Oracle& o, const uint64_t* chain, uint64_t nb, uint32_t L, float ttft_target,
            float tpot_target, Row& row, WminOverride ov = WminOverride()) {
  const orc_model& m = o.m;
  const uint32_t I = o.I;
  row.hit.assign(I, 0); row.tpot.assign(I, 0.f); row.ttft.assign(I, 0.f); row.cls.assign(I, 3);
  row.pick = -1; row.path = 2;
  const float Lf = (float)L;
  const float t_cached = t_pf(m, 0.0f, Lf);       // fully cached input
  const float t_cold = t_pf(m, Lf, 0.0f);         // fully uncached input
  const float Z = t_cold - t_cached;              // CacheBenefit (Alg. 1, Section 6.1)
  const float etaZ = m.eta * Z;
  const float ttft_budget = t_cold > ttft_target ? t_cold : ttft_target;
  std::vector<float> W(I, 0.f), tpf(I, 0.f);
  std::vector<int64_t> n_tok(I, 0);
  std::vector<char> inA(I, 0);
  bool anyA = false;
  float Wmin = 0.f;
  // Capacity guard + RecomputeCost (Alg. 1, KVC-first filtering; Section 6.1).
  for (uint32_t i = 0; i < I; ++i) {
    const orc_inst& s = o.st[i];
    uint64_t h = hit_len(o, i, chain, nb);
    row.hit[i] = h;
    int64_t c = 16 * (int64_t)h;
    int64_t n = (int64_t)L - c;
    n_tok[i] = n;
    tpf[i] = t_pf(m, (float)n, (float)c);
    W[i] = tpf[i] - t_cached;
    inA[i] = ((int64_t)s.b + s.qr + 1 <= (int64_t)s.B_max) && (s.S + (int64_t)L <= s.M_KV);
    if (inA[i]) {
      if (!anyA || W[i] < Wmin) Wmin = W[i];
      anyA = true;
    }
    // Predicted latencies for every instance (Eq. 4, Eq. 7, Eq. 9 / configuration form).
    const int64_t Bp = (int64_t)s.b + s.qr + 1;
    const int64_t Sp = s.S + (int64_t)L;
    const float f = ema_factor(m, Bp);
    float dec = m.b0 + m.b1 * (float)Bp;
    dec = dec + m.b2 * (float)Sp;
    dec = dec * f;
    float tp;
    if (m.interference_mode == 0) {
      tp = dec + m.g_q * (float)(s.q + n);
    } else {
      const float den = m.lout_median > 1.0f ? m.lout_median : 1.0f;
      const float interf = ((int64_t)s.b + s.qr > 0) ? tpf[i] / den : 0.0f;
      tp = dec + interf;
    }
    const float tq = m.a0 * (float)s.qr + m.a1 * (float)s.q;
    row.tpot[i] = tp;
    row.ttft[i] = tpf[i] + tq;
  }
  row.anyA = anyA;
  row.Wmin = Wmin;
  if (!anyA) return;  // Reject (Alg. 1: A empty)
  if (ov.given) Wmin = ov.Wmin;
  // Normalised recompute filter, Eq. 8; SLO admission (Alg. 1 TPOT filter, plus TTFT budget).
  bool anyT = false;
  for (uint32_t i = 0; i < I; ++i) {
    if (!inA[i]) continue;
    bool inC = (Z > 0.0f) ? ((W[i] - Wmin) <= etaZ) : true;
    if (!m.cache_filter) inC = true;
    if (!inC) { row.cls[i] = 2; continue; }
    bool ok = row.tpot[i] < tpot_target;
    if (m.ttft_filter) ok = ok && (row.ttft[i] <= ttft_budget);
    if (!m.slo_filter) ok = true;
    row.cls[i] = ok ? 0 : 1;
    anyT = anyT || ok;
  }
  // Instance order (Section 6.2, Table 4): D more decoding requests, C more cached blocks, Q fewer
  // queued requests, H smaller predicted TPOT headroom (target - TPOT); the lowest id last.
  auto before = [&](uint32_t i, uint32_t z, int32_t sel) -> bool {
    const orc_inst& a = o.st[i];
    const orc_inst& y = o.st[z];
    if (sel == 5) {
      const float ha = tpot_target - row.tpot[i], hy = tpot_target - row.tpot[z];
      if (ha != hy) return ha < hy;
      if (row.hit[i] != row.hit[z]) return row.hit[i] > row.hit[z];
      return a.qr < y.qr;
    }
    if (a.b != y.b) return a.b > y.b;
    const bool useC = sel == 0 || sel == 3 || sel == 4, useQ = sel == 0 || sel == 2 || sel == 4;
    const bool c_first = sel != 4;
    if (c_first) {
      if (useC && row.hit[i] != row.hit[z]) return row.hit[i] > row.hit[z];
      if (useQ && a.qr != y.qr) return a.qr < y.qr;
    } else {
      if (useQ && a.qr != y.qr) return a.qr < y.qr;
      if (useC && row.hit[i] != row.hit[z]) return row.hit[i] > row.hit[z];
    }
    return false;  // equal: the lower id, visited first, stays
  };
  int32_t best = -1;
  if (anyT) {
    for (uint32_t i = 0; i < I; ++i) {
      if (row.cls[i] != 0) continue;
      if (best < 0 || before(i, (uint32_t)best, m.selector)) best = (int32_t)i;
    }
    row.pick = best; row.path = 0;
  } else if (m.fallback == 1) {
    // The ablations' D-C-Q fallback over C (Table 3, configurations T and CT).
    for (uint32_t i = 0; i < I; ++i) {
      if (row.cls[i] != 1) continue;
      if (best < 0 || before(i, (uint32_t)best, 0)) best = (int32_t)i;
    }
    row.pick = best; row.path = best >= 0 ? 1 : 2;
  } else {
    // CacheAwareLB = LMetric over C: pending uncached prefill tokens x active requests,
    // both including the arriving request.
    uint64_t bestv = 0;
    for (uint32_t i = 0; i < I; ++i) {
      if (row.cls[i] != 1) continue;
      const orc_inst& s = o.st[i];
      uint64_t v = (uint64_t)(s.q + n_tok[i]) * (uint64_t)((int64_t)s.b + s.qr + 1);
      if (best < 0 || v < bestv) { best = (int32_t)i; bestv = v; }
    }
    row.pick = best; row.path = best >= 0 ? 1 : 2;
  }
}

void touch_block(Oracle& o, uint32_t i, uint64_t h, uint32_t last_use) {
  auto it = o.meta[i].find(h);
  if (it == o.meta[i].end() || it->second.last_use >= last_use) return;
  if (it->second.children == 0) {
    o.leaves[i].erase({it->second.last_use, h});
    o.leaves[i].insert({last_use, h});
  }
  it->second.last_use = last_use;
}

void insert_block(Oracle& o, uint32_t i, uint64_t h, uint64_t parent, uint32_t last_use) {
  bool added = o.cache[i].insert(h).second;
  if (!o.track) return;
  auto& mm = o.meta[i];
  if (added) {
    mm[h] = BlockMeta{parent, 0, last_use};
    o.leaves[i].insert({last_use, h});
    if (parent) {
      auto it = mm.find(parent);
      if (it != mm.end()) {
        if (it->second.children == 0) o.leaves[i].erase({it->second.last_use, parent});
        it->second.children += 1;
      }
    }
  } else {
    touch_block(o, i, h, last_use);
  }
}

// Leaf-first LRU eviction down to the instance's capacity.
void evict_to_cap(Oracle& o, uint32_t i) {
  while (o.cache[i].size() > o.cap[i] && !o.leaves[i].empty()) {
    const auto victim = *o.leaves[i].begin();
    o.leaves[i].erase(o.leaves[i].begin());
    const uint64_t h = victim.second;
    const uint64_t parent = o.meta[i][h].parent;
    o.meta[i].erase(h);
    o.cache[i].erase(h);
    if (parent) {
      auto it = o.meta[i].find(parent);
      if (it != o.meta[i].end()) {
        it->second.children -= 1;
        if (it->second.children == 0) o.leaves[i].insert({it->second.last_use, parent});
      }
    }
  }
}

}  // namespace

extern "C" {

void* orc_create(uint32_t I, const orc_model* m, int32_t track_lru) {
  if (!m || m->nseg < 1 || m->nseg > 16) return nullptr;
  Oracle* o = new Oracle();
  o->I = I;
  o->m = *m;
  o->cache.resize(I);
  o->st.assign(I, orc_inst{0, 0, 0, 0, 0, 0});
  o->track = track_lru != 0;
  if (o->track) {
    o->meta.resize(I);
    o->leaves.resize(I);
  }
  o->queue.resize(I);
  o->decoding.resize(I);
  o->cap.assign(I, UINT64_MAX);
  return o;
}

void orc_destroy(void* h) { delete static_cast<Oracle*>(h); }

void orc_reserve(void* h, uint32_t inst, uint64_t n) {
  Oracle* o = static_cast<Oracle*>(h);
  o->cache[inst].reserve(n);
  if (o->track) o->meta[inst].reserve(n);
}

// Insert n chained blocks into instance inst: block 0's parent is `parent` (0 = root), block k's
// parent is block k-1.
void orc_insert_chain(void* h, uint32_t inst, const uint64_t* chain, uint64_t n, uint64_t parent,
                      uint32_t last_use) {
  Oracle* o = static_cast<Oracle*>(h);
  for (uint64_t k = 0; k < n; ++k) insert_block(*o, inst, chain[k], k ? chain[k - 1] : parent, last_use);
}

// Bulk form of the above over a CSR of chains.
void orc_insert_chains(void* h, uint64_t nchains, const uint32_t* inst, const uint64_t* off,
                       const uint64_t* hash, const uint64_t* parent, uint32_t last_use) {
  for (uint64_t c = 0; c < nchains; ++c)
    orc_insert_chain(h, inst[c], hash + off[c], off[c + 1] - off[c], parent[c], last_use);
}

uint64_t orc_cached_blocks(void* h, uint32_t inst) {
  return static_cast<Oracle*>(h)->cache[inst].size();
}

int32_t orc_contains(void* h, uint32_t inst, uint64_t block) {
  return static_cast<Oracle*>(h)->cache[inst].count(block) ? 1 : 0;
}

void orc_set_state(void* h, const orc_inst* s) {
  Oracle* o = static_cast<Oracle*>(h);
  std::memcpy(o->st.data(), s, sizeof(orc_inst) * o->I);
}

void orc_get_state(void* h, orc_inst* s) {
  Oracle* o = static_cast<Oracle*>(h);
  std::memcpy(s, o->st.data(), sizeof(orc_inst) * o->I);
}

uint64_t orc_hit(void* h, uint32_t inst, const uint64_t* chain, uint64_t nb) {
  return hit_len(*static_cast<Oracle*>(h), inst, chain, nb);
}

// Hit lengths of selected (request, instance) pairs.
void orc_hit_pairs(void* h, const uint64_t* off, const uint64_t* hash, uint64_t npairs,
                   const uint32_t* req, const uint32_t* inst, uint32_t* out) {
  Oracle* o = static_cast<Oracle*>(h);
  for (uint64_t k = 0; k < npairs; ++k) {
    const uint64_t* ch = hash + off[req[k]];
    out[k] = (uint32_t)hit_len(*o, inst[k], ch, off[req[k] + 1] - off[req[k]]);
  }
}

// Score mode: each listed request against the current state, independently (no state change).
// Outputs are row-major [nrows x I]; any output pointer may be null.
void orc_score_rows(void* h, const uint64_t* off, const uint64_t* hash, const uint32_t* L,
                    const float* ttft_target, const float* tpot_target, uint64_t nrows,
                    const uint32_t* rows, uint32_t* hits, float* tpot, float* ttft, uint8_t* cls,
                    int32_t* best, uint8_t* path) {
  Oracle* o = static_cast<Oracle*>(h);
  Row row;
  for (uint64_t k = 0; k < nrows; ++k) {
    uint32_t r = rows[k];
    decide(*o, hash + off[r], off[r + 1] - off[r], L[r], ttft_target[r], tpot_target[r], row);
    for (uint32_t i = 0; i < o->I; ++i) {
      size_t x = (size_t)k * o->I + i;
      if (hits) hits[x] = (uint32_t)row.hit[i];
      if (tpot) tpot[x] = row.tpot[i];
      if (ttft) ttft[x] = row.ttft[i];
      if (cls) cls[x] = row.cls[i];
    }
    if (best) best[k] = row.pick;
    if (path) path[k] = row.path;
  }
}

// Score mode over one column block of an instance pool (the oracle holds the block's instances):
// wmin_out / anyA_out (nullable) receive W_min over the block's A and whether A is not empty;
// with wmin_in non-null, row k's recompute filter uses W_min = wmin_in[k] (the pool's W_min; not read
// where the block's A is empty) instead of the block's own.  Other outputs as
// orc_score_rows; best is the block's pick (a block-local id).
void orc_score_rows_block(void* h, const uint64_t* off, const uint64_t* hash, const uint32_t* L,
                          const float* ttft_target, const float* tpot_target, uint64_t nrows,
                          const uint32_t* rows, const float* wmin_in, float* wmin_out, uint8_t* anyA_out,
                          uint32_t* hits, uint8_t* cls, int32_t* best, uint8_t* path) {
  Oracle* o = static_cast<Oracle*>(h);
  Row row;
  for (uint64_t k = 0; k < nrows; ++k) {
    uint32_t r = rows[k];
    WminOverride ov;
    if (wmin_in) { ov.given = true; ov.Wmin = wmin_in[k]; }
    decide(*o, hash + off[r], off[r + 1] - off[r], L[r], ttft_target[r], tpot_target[r], row, ov);
    if (wmin_out) wmin_out[k] = row.Wmin;
    if (anyA_out) anyA_out[k] = row.anyA ? 1 : 0;
    for (uint32_t i = 0; i < o->I; ++i) {
      if (hits) hits[(size_t)k * o->I + i] = (uint32_t)row.hit[i];
      if (cls) cls[(size_t)k * o->I + i] = row.cls[i];
    }
    if (best) best[k] = row.pick;
    if (path) path[k] = row.path;
  }
}

// Greedy in-window assignment: requests in arrival order, each decided by Algorithm 1 on the
// state left by all earlier decisions; an admitted request adds qr += 1, q += n, S += L on its
// instance and its uncached blocks chain[h..nb) to that instance's cache.  `hit_chosen` receives
// the hit length on the chosen instance (0 on reject).  window_id stamps LRU use times.
void orc_schedule(void* h, uint32_t R, const uint64_t* off, const uint64_t* hash, const uint32_t* L,
                  const float* ttft_target, const float* tpot_target, const uint32_t* out_tokens,
                  int32_t* assign, uint8_t* path, uint32_t* hit_chosen, uint32_t window_id) {
  Oracle* o = static_cast<Oracle*>(h);
  Row row;
  for (uint32_t r = 0; r < R; ++r) {
    const uint64_t* ch = hash + off[r];
    const uint64_t nb = off[r + 1] - off[r];
    decide(*o, ch, nb, L[r], ttft_target[r], tpot_target[r], row);
    if (assign) assign[r] = row.pick;
    if (path) path[r] = row.path;
    if (hit_chosen) hit_chosen[r] = row.pick >= 0 ? (uint32_t)row.hit[row.pick] : 0;
    if (row.pick < 0) continue;
    const uint32_t j = (uint32_t)row.pick;
    const uint64_t hj = row.hit[j];
    orc_inst& s = o->st[j];
    s.qr += 1;
    s.q += (int64_t)L[r] - 16 * (int64_t)hj;
    s.S += (int64_t)L[r];
    if (o->track)
      for (uint64_t k = 0; k < hj; ++k) touch_block(*o, j, ch[k], window_id);
    for (uint64_t k = hj; k < nb; ++k) insert_block(*o, j, ch[k], k ? ch[k - 1] : 0, window_id);
    if (out_tokens)
      o->queue[j].push_back(Oracle::Queued{L[r], out_tokens[r], (uint64_t)((int64_t)L[r] - 16 * (int64_t)hj)});
  }
}

// Cache capacities for eviction (blocks per instance).
void orc_set_capacity(void* h, const uint64_t* cap) {
  Oracle* o = static_cast<Oracle*>(h);
  for (uint32_t i = 0; i < o->I; ++i) o->cap[i] = cap[i];
}

// Requests in flight at the start of a stream.  state 0: queued (FIFO in the given order, rem =
// remaining prefill tokens), 1: decoding (rem = remaining output tokens).  The instance state's
// b, qr, q and S are recomputed from them (S = sum of queued L + decoding L + emitted tokens).
void orc_load_requests(void* h, uint64_t n, const uint32_t* inst, const uint32_t* state, const uint32_t* L,
                       const uint32_t* out, const uint64_t* rem) {
  Oracle* o = static_cast<Oracle*>(h);
  for (uint32_t i = 0; i < o->I; ++i) {
    o->queue[i].clear();
    o->decoding[i].clear();
    o->st[i].b = 0; o->st[i].qr = 0; o->st[i].q = 0; o->st[i].S = 0;
  }
  for (uint64_t k = 0; k < n; ++k) {
    orc_inst& s = o->st[inst[k]];
    if (state[k] == 0) {
      o->queue[inst[k]].push_back(Oracle::Queued{L[k], out[k], rem[k]});
      s.qr += 1;
      s.q += (int64_t)rem[k];
      s.S += (int64_t)L[k];
    } else {
      o->decoding[inst[k]].push_back(Oracle::Decoding{L[k], out[k], (uint32_t)rem[k]});
      s.b += 1;
      s.S += (int64_t)L[k] + (int64_t)(out[k] - (uint32_t)rem[k]);
    }
  }
}

// One window of engine progress, then eviction to capacity (see the header).
void orc_advance(void* h, float window_ms, uint64_t prefill_tokens, int32_t evict) {
  Oracle* o = static_cast<Oracle*>(h);
  const orc_model& m = o->m;
  for (uint32_t i = 0; i < o->I; ++i) {
    orc_inst& s = o->st[i];
    float t_iter = m.b0 + m.b1 * (float)s.b;
    t_iter = t_iter + m.b2 * (float)s.S;
    const float per = window_ms / t_iter;
    int64_t k = (int64_t)per;  // per > 0: truncation is floor
    if (k < 1) k = 1;
    std::vector<Oracle::Decoding> keep;
    for (auto& d : o->decoding[i]) {
      const uint32_t e = (uint64_t)d.rem < (uint64_t)k ? d.rem : (uint32_t)k;
      d.rem -= e;
      s.S += e;
      if (d.rem == 0) {
        s.b -= 1;
        s.S -= (int64_t)d.L + (int64_t)d.out;
      } else {
        keep.push_back(d);
      }
    }
    o->decoding[i].swap(keep);
    uint64_t budget = prefill_tokens;
    while (budget > 0 && !o->queue[i].empty()) {
      Oracle::Queued& qd = o->queue[i].front();
      const uint64_t d = qd.rem < budget ? qd.rem : budget;
      qd.rem -= d;
      s.q -= (int64_t)d;
      budget -= d;
      if (qd.rem == 0) {
        o->decoding[i].push_back(Oracle::Decoding{qd.L, qd.out, qd.out});
        o->queue[i].pop_front();
        s.qr -= 1;
        s.b += 1;
      }
    }
    if (evict && o->track) evict_to_cap(*o, i);
  }
}

uint32_t orc_last_use(void* h, uint32_t inst, uint64_t block) {
  Oracle* o = static_cast<Oracle*>(h);
  if (!o->track) return 0;
  auto it = o->meta[inst].find(block);
  return it == o->meta[inst].end() ? 0 : it->second.last_use;
}

// Online calibration (Section 5.3): per decode-batch segment a multiplicative EMA factor of the
// decode term.  Each pure-decode feedback sample (measured batch size B, total context S, measured
// forward duration) is taken in order: the base model's prediction at the same B and S is
// (b0 + b1 B) + b2 S, the measured-to-predicted ratio is clipped to [0.5, 2], the factor of B's
// segment moves by the update weight towards it, f <- f + weight (ratio - f), and is clipped to
// [1, 2].  Factors start at 1 (the model's table as given).
void orc_calibrate(void* h, uint64_t n, const int32_t* batch, const int64_t* ctx_tokens, const float* measured_ms,
                   float weight) {
  Oracle* o = static_cast<Oracle*>(h);
  orc_model& m = o->m;
  for (uint64_t k = 0; k < n; ++k) {
    const int64_t B = batch[k];
    float base = m.b0 + m.b1 * (float)B;
    base = base + m.b2 * (float)ctx_tokens[k];
    float ratio = measured_ms[k] / base;
    if (ratio < 0.5f) ratio = 0.5f;
    if (ratio > 2.0f) ratio = 2.0f;
    int s = 0;
    for (int q = 0; q < m.nseg; ++q)
      if ((int64_t)m.seg_lo[q] <= B) s = q;
    float f = m.ema_factor[s] + weight * (ratio - m.ema_factor[s]);
    if (f < 1.0f) f = 1.0f;
    if (f > 2.0f) f = 2.0f;
    m.ema_factor[s] = f;
  }
}

void orc_ema_factors(void* h, float* out) {
  const Oracle* o = static_cast<const Oracle*>(h);
  for (int s = 0; s < 16; ++s) out[s] = o->m.ema_factor[s];
}

}  // extern "C"
