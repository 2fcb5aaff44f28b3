// Seeded synthetic workload generator for the scheduler hot path.
//
// Produces, for one scheduling window: the requests (token-prefix block-hash chains in CSR form,
// prompt lengths, TTFT/TPOT targets) and the instances (cached chains, decode batch, queued
// prefill, KV tokens, limits).  It holds none of the scheduler's arithmetic: no hit lengths, no
// latency model, no filters.  Both the oracle and the CUDA path consume its arrays.
//
// Determinism: every random draw comes from a splitmix64 stream keyed by (seed, purpose, id), and
// the only floating-point work (lognormal increments, Zipf weights) uses + - * / in double with
// -ffp-contract=off plus the series below, never libm, so x86-64 and aarch64 builds produce
// bit-identical workloads.
//
// Session model (stands in for the production agentic trace of the paper's Table 2, which is not
// available): a session is an endless series of episodes.  An episode starts a fresh token branch
// that shares only the system prompt, has U{steps_lo..steps_hi} steps, starts at a prompt length
// U{ctx_min..ctx_start_hi} and grows by lognormal(inc_mu, inc_sigma) tokens per step; it ends early
// when the next prompt would exceed ctx_max (context compaction).  Step k+1's prompt extends step
// k's (the paper's Section 1 request chains with long shared prefixes).  With fork_every > 0, every
// fork_every-th step branches from the prompt of fork_every/2 steps earlier.

#include <cstdint>
#include <cstring>
#include <cstdlib>
#include <vector>
#include <map>
#include <algorithm>

namespace {

constexpr uint64_t kGolden = 0x9E3779B97F4A7C15ULL;

// splitmix64 (Steele, Lea and Flood, OOPSLA 2014): the state advances by the golden-ratio
// increment, the output is the two-round xor-shift-multiply finaliser of the new state.
inline uint64_t sm_finalise(uint64_t z) {
  z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ULL;
  z = (z ^ (z >> 27)) * 0x94D049BB133111EBULL;
  return z ^ (z >> 31);
}
// One generator step taken from state x (the value splitmix64 returns when seeded with x).
inline uint64_t splitmix64(uint64_t x) { return sm_finalise(x + kGolden); }

enum Purpose : uint64_t {
  kPurposeSession = 1, kPurposePlace = 2, kPurposeHome = 3, kPurposePick = 4, kPurposeState = 5,
  kPurposeFill = 6, kPurposeFillTarget = 7, kPurposeBranchKey = 8, kPurposeSysKey = 9,
  kPurposeOutput = 10, kPurposeRequests = 11,
};

struct Rng {
  uint64_t s;
  Rng(uint64_t seed, uint64_t purpose, uint64_t id) {
    s = splitmix64(splitmix64(splitmix64(seed) ^ purpose) ^ id);
  }
  uint64_t next() { s += kGolden; return sm_finalise(s); }
  double unit() { return (double)(next() >> 11) * (1.0 / 9007199254740992.0); }
  uint64_t below(uint64_t n) { return (uint64_t)(((unsigned __int128)next() * n) >> 64); }
  int64_t range(int64_t lo, int64_t hi) { return lo + (int64_t)below((uint64_t)(hi - lo + 1)); }
  // Irwin-Hall: the sum of 12 uniforms minus 6 is a standard-normal stand-in on [-6, 6].
  double normal() { double a = 0.0; for (int k = 0; k < 12; ++k) a = a + unit(); return a - 6.0; }
};

// e^x by range reduction x = k ln2 + r, |r| <= ln2/2, and a 24-term Taylor series of e^r.
double det_exp(double x) {
  const double ln2 = 0.6931471805599453;
  double kf = x / ln2;
  int64_t k = (int64_t)(kf < 0.0 ? kf - 0.5 : kf + 0.5);
  double r = x - (double)k * ln2;
  double term = 1.0, sum = 1.0;
  for (int n = 1; n < 24; ++n) { term = term * r / (double)n; sum = sum + term; }
  if (k < -1000) return 0.0;
  if (k > 1000) k = 1000;
  uint64_t bits = (uint64_t)(k + 1023) << 52;
  double p; std::memcpy(&p, &bits, 8);
  return sum * p;
}

// ln x for x > 0 (normal): x = m 2^e with m in [1/sqrt2, sqrt2], ln m = 2 atanh((m-1)/(m+1)).
double det_log(double x) {
  uint64_t bits; std::memcpy(&bits, &x, 8);
  int64_t e = (int64_t)((bits >> 52) & 0x7FF) - 1023;
  bits = (bits & 0x000FFFFFFFFFFFFFULL) | 0x3FF0000000000000ULL;
  double m; std::memcpy(&m, &bits, 8);
  if (m > 1.4142135623730951) { m = m * 0.5; e += 1; }
  double y = (m - 1.0) / (m + 1.0), y2 = y * y, term = y, sum = 0.0;
  for (int n = 1; n < 40; n += 2) { sum = sum + term / (double)n; term = term * y2; }
  return 2.0 * sum + (double)e * 0.6931471805599453;
}

}  // namespace

extern "C" {

// Parameters of one synthetic workload (all lengths in tokens unless noted).
typedef struct {
  uint64_t seed;
  uint32_t num_instances, window_requests;
  uint32_t num_sessions;
  uint32_t steps_lo, steps_hi;      // steps per episode
  double inc_mu, inc_sigma;         // lognormal prompt growth per step
  uint32_t ctx_min, ctx_start_hi;   // first prompt of an episode ~ U{ctx_min..ctx_start_hi}
  uint32_t ctx_max;                 // prompts never exceed this
  uint32_t sys_tokens;              // shared system prompt (multiple of 16)
  double zipf_s;                    // session popularity exponent; 0 = uniform
  double affinity;                  // probability a history step runs on the session's home
  uint32_t fork_every;              // 0 = no forks
  uint32_t hist_lo, hist_hi;        // history steps per session before the first window
  uint64_t cap_blocks;              // per-instance cache capacity (blocks)
  double fill_lo, fill_hi;          // cached blocks = U[fill_lo, fill_hi] x cap_blocks
  uint32_t b_hi;                    // decode batch ~ U{0..b_hi}
  uint64_t q_hi;                    // queued prefill tokens ~ U{0..q_hi}
  uint32_t b_max;                   // decode-slot limit
  float tpot_target_ms, ttft_target_ms;
  double out_mu, out_sigma;         // output length lognormal (streaming windows)
  uint32_t out_lo, out_hi;          // output length clamp
  uint32_t kv_rule;                 // 0: S = cached session tokens; 1: also <= M_KV * b / b_max
} ws_params;

}  // extern "C"

namespace {

struct Branch {
  int64_t parent;                 // -1: no parent
  uint64_t fork_pos;              // tokens [0, fork_pos) are the parent's
  uint64_t fork_blk;              // first block this branch owns = fork_pos / 16
  uint64_t key;                   // token stream key
  std::vector<uint64_t> own;      // chain hashes of blocks [fork_blk, fork_blk + own.size())
};

struct Session {
  Rng rng;
  uint32_t home;
  int64_t branch = -1;            // current branch
  uint32_t step = 0, steps = 0;   // step within episode, episode length
  uint64_t len = 0;               // current prompt length
  std::vector<uint64_t> lens;     // prompt lengths of this episode's steps
  uint64_t episode = 0;
  explicit Session(const Rng& r) : rng(r), home(0) {}
};

struct Request { int64_t branch; uint64_t len; uint32_t session; uint32_t out; };

struct Gen {
  ws_params p;
  std::vector<Branch> br;
  int64_t sys_branch = -1;
  std::vector<Session> sess;
  std::vector<double> zipf_cdf;
  Rng pick_rng;
  uint64_t windows_made = 0;

  // current window
  std::vector<uint64_t> w_off, w_hash;
  std::vector<uint32_t> w_len, w_sess, w_out;
  std::vector<float> w_ttft, w_tpot;

  // instances
  std::vector<int32_t> s_b, s_qr, s_bmax;
  std::vector<int64_t> s_q, s_S, s_M;
  std::vector<uint64_t> s_cap;
  std::vector<uint32_t> c_inst;
  std::vector<uint64_t> c_off, c_hash, c_parent;

  explicit Gen(const ws_params& q) : p(q), pick_rng(q.seed, kPurposePick, 0) {}

  uint32_t token(int64_t b, uint64_t pos) const {
    while (br[b].parent >= 0 && pos < br[b].fork_pos) b = br[b].parent;
    return (uint32_t)(splitmix64(br[b].key + pos) & 0x1FFFFu);
  }
  uint64_t chain_at(int64_t b, uint64_t k) const {
    while (k < br[b].fork_blk) b = br[b].parent;
    return br[b].own[k - br[b].fork_blk];
  }
  // Extend branch b's chain to nblk blocks: x_0 = 0, x <- splitmix64(x ^ token) per token, a block's
  // hash is x after its 16th token (0 remapped to 1), and that stored value continues the chain.
  void ensure(int64_t b, uint64_t nblk) {
    if (br[b].parent >= 0 && br[b].fork_blk > 0) ensure(br[b].parent, std::min(nblk, br[b].fork_blk));
    if (nblk <= br[b].fork_blk) return;
    while (br[b].fork_blk + br[b].own.size() < nblk) {
      uint64_t k = br[b].fork_blk + br[b].own.size();
      uint64_t x = k ? chain_at(b, k - 1) : 0;
      for (uint64_t j = 0; j < 16; ++j) {
        x = splitmix64(x ^ (uint64_t)token(b, 16 * k + j));
      }
      if (x == 0) x = 1;
      br[b].own.push_back(x);
    }
  }
  int64_t new_branch(int64_t parent, uint64_t fork_pos) {
    Branch nb;
    nb.parent = parent;
    nb.fork_pos = parent >= 0 ? fork_pos : 0;
    nb.fork_blk = nb.fork_pos / 16;
    nb.key = splitmix64(splitmix64(p.seed ^ 0xB4A7C0DEULL) + (uint64_t)br.size() * kGolden) ^ kPurposeBranchKey;
    br.push_back(std::move(nb));
    return (int64_t)br.size() - 1;
  }
  uint64_t lognormal_tokens(Rng& r, double mu, double sigma) {
    double v = det_exp(mu + sigma * r.normal());
    if (v < 1.0) v = 1.0;
    if (v > 1e9) v = 1e9;
    return (uint64_t)(v + 0.5);
  }
  void new_episode(Session& s) {
    s.episode += 1;
    s.branch = new_branch(sys_branch, p.sys_tokens);
    s.steps = (uint32_t)s.rng.range(p.steps_lo, p.steps_hi);
    s.step = 1;
    uint64_t lo = std::max<uint64_t>(p.ctx_min, p.sys_tokens);
    uint64_t hi = std::max<uint64_t>(lo, p.ctx_start_hi);
    s.len = (uint64_t)s.rng.range((int64_t)lo, (int64_t)hi);
    if (s.len > p.ctx_max) s.len = p.ctx_max;
    s.lens.assign(1, s.len);
  }
  // Advance session s by one step and return (branch, prompt length).
  void advance(Session& s) {
    if (s.branch < 0) { new_episode(s); return; }
    uint64_t inc = lognormal_tokens(s.rng, p.inc_mu, p.inc_sigma);
    if (s.step >= s.steps || s.len + inc > p.ctx_max) { new_episode(s); return; }
    s.step += 1;
    s.len += inc;
    if (p.fork_every && s.step % p.fork_every == 0 && s.lens.size() > p.fork_every / 2) {
      uint64_t fork_pos = s.lens[s.lens.size() - 1 - p.fork_every / 2];
      if (fork_pos > p.sys_tokens) s.branch = new_branch(s.branch, fork_pos);
    }
    s.lens.push_back(s.len);
  }
  uint32_t pick_session() {
    if (p.zipf_s <= 0.0) return (uint32_t)pick_rng.below(p.num_sessions);
    double u = pick_rng.unit() * zipf_cdf.back();
    size_t k = (size_t)(std::upper_bound(zipf_cdf.begin(), zipf_cdf.end(), u) - zipf_cdf.begin());
    return (uint32_t)std::min<size_t>(k, p.num_sessions - 1);
  }
  // Blocks shared by the chains of branches a and b (both extended far enough).
  uint64_t common_blocks(int64_t a, int64_t b) const {
    std::map<int64_t, uint64_t> up;  // ancestor of a -> min fork block on the path from a
    uint64_t m = UINT64_MAX;
    for (int64_t x = a; x >= 0; x = br[x].parent) {
      up[x] = m;
      if (br[x].parent >= 0) m = std::min(m, br[x].fork_blk);
    }
    m = UINT64_MAX;
    for (int64_t x = b; x >= 0; x = br[x].parent) {
      auto it = up.find(x);
      if (it != up.end()) return std::min(m, it->second);
      if (br[x].parent >= 0) m = std::min(m, br[x].fork_blk);
    }
    return 0;
  }

  void build() {
    if (p.sys_tokens > 0) {
      sys_branch = new_branch(-1, 0);
      br[sys_branch].key = splitmix64(p.seed ^ kPurposeSysKey);
    }
    if (p.zipf_s > 0.0) {
      zipf_cdf.resize(p.num_sessions);
      double acc = 0.0;
      for (uint32_t k = 0; k < p.num_sessions; ++k) {
        acc = acc + det_exp(-p.zipf_s * det_log((double)(k + 1)));
        zipf_cdf[k] = acc;
      }
    }
    const uint32_t I = p.num_instances;
    sess.reserve(p.num_sessions);
    for (uint32_t s = 0; s < p.num_sessions; ++s) {
      sess.emplace_back(Rng(p.seed, kPurposeSession, s));
      sess.back().home = (uint32_t)Rng(p.seed, kPurposeHome, s).below(I);
    }
    // History: each session served hist steps; the serving instance caches that step's prompt.
    std::vector<std::map<int64_t, uint64_t>> cached(I);  // instance -> branch -> cached blocks
    for (uint32_t s = 0; s < p.num_sessions; ++s) {
      Rng place(p.seed, kPurposePlace, s);
      uint32_t hist = (uint32_t)place.range(p.hist_lo, p.hist_hi);
      for (uint32_t h = 0; h < hist; ++h) {
        advance(sess[s]);
        uint32_t inst = place.unit() < p.affinity ? sess[s].home : (uint32_t)place.below(I);
        uint64_t nblk = sess[s].len / 16;
        uint64_t& slot = cached[inst][sess[s].branch];
        slot = std::max(slot, nblk);
      }
    }
    // Instance contents: union of cached prefixes (each shared block emitted once, parent first),
    // trimmed to the fill target, then random chains up to it.
    s_b.resize(I); s_qr.resize(I); s_bmax.resize(I); s_q.resize(I); s_S.resize(I); s_M.resize(I);
    s_cap.assign(I, p.cap_blocks);
    c_off.assign(1, 0);
    for (uint32_t i = 0; i < I; ++i) {
      Rng ft(p.seed, kPurposeFillTarget, i);
      double frac = p.fill_lo + (p.fill_hi - p.fill_lo) * ft.unit();
      uint64_t target = (uint64_t)(frac * (double)p.cap_blocks);
      if (target > p.cap_blocks) target = p.cap_blocks;
      uint64_t used = 0, session_tokens = 0;
      std::vector<std::pair<int64_t, uint64_t>> done;  // emitted (branch, blocks)
      auto emit = [&](int64_t b, uint64_t nblk) {
        uint64_t start = 0;
        for (auto& e : done) start = std::max(start, std::min(common_blocks(b, e.first), std::min(e.second, nblk)));
        if (start >= nblk) return nblk;
        uint64_t take = std::min(nblk - start, target - used);
        if (take == 0) return start;
        ensure(b, start + take);
        c_inst.push_back(i);
        c_parent.push_back(start ? chain_at(b, start - 1) : 0);
        for (uint64_t k = start; k < start + take; ++k) c_hash.push_back(chain_at(b, k));
        c_off.push_back(c_hash.size());
        used += take;
        done.emplace_back(b, start + take);
        return start + take;
      };
      for (auto& kv : cached[i]) {
        if (used >= target) break;
        uint64_t got = emit(kv.first, kv.second);
        session_tokens += 16 * got;
      }
      Rng fr(p.seed, kPurposeFill, i);
      while (used < target) {
        uint64_t n = std::min<uint64_t>((uint64_t)fr.range(64, 512), target - used);
        c_inst.push_back(i);
        c_parent.push_back(0);
        for (uint64_t k = 0; k < n; ++k) {
          uint64_t h = fr.next();
          c_hash.push_back(h ? h : 1);
        }
        c_off.push_back(c_hash.size());
        used += n;
      }
      Rng st(p.seed, kPurposeState, i);
      s_b[i] = (int32_t)st.range(0, p.b_hi);
      s_q[i] = (int64_t)st.range(0, (int64_t)p.q_hi);
      s_qr[i] = (int32_t)((s_q[i] + 4095) / 4096);
      s_M[i] = (int64_t)(16 * p.cap_blocks);
      int64_t kv = std::min<int64_t>((int64_t)session_tokens, s_M[i]);
      if (p.kv_rule == 1 && p.b_max > 0) kv = std::min<int64_t>(kv, s_M[i] * s_b[i] / (int64_t)p.b_max);
      s_S[i] = kv;
      s_bmax[i] = (int32_t)p.b_max;
    }
  }

  void make_window(uint32_t R) {
    w_off.assign(1, 0); w_hash.clear(); w_len.clear(); w_sess.clear(); w_out.clear();
    w_ttft.clear(); w_tpot.clear();
    Rng outr(p.seed, kPurposeOutput, windows_made);
    for (uint32_t r = 0; r < R; ++r) {
      uint32_t s = pick_session();
      advance(sess[s]);
      uint64_t nblk = sess[s].len / 16;
      ensure(sess[s].branch, nblk);
      for (uint64_t k = 0; k < nblk; ++k) w_hash.push_back(chain_at(sess[s].branch, k));
      w_off.push_back(w_hash.size());
      w_len.push_back((uint32_t)sess[s].len);
      w_sess.push_back(s);
      uint64_t o = lognormal_tokens(outr, p.out_mu, p.out_sigma);
      o = std::max<uint64_t>(p.out_lo, std::min<uint64_t>(p.out_hi, o));
      w_out.push_back((uint32_t)o);
      w_ttft.push_back(p.ttft_target_ms);
      w_tpot.push_back(p.tpot_target_ms);
    }
    windows_made += 1;
  }
};

}  // namespace

extern "C" {

void* ws_generate(const ws_params* p) {
  if (!p || p->num_instances == 0 || p->num_sessions == 0 || p->steps_lo == 0 ||
      p->steps_hi < p->steps_lo || p->ctx_max < 16 || (p->sys_tokens % 16) != 0) return nullptr;
  Gen* g = new Gen(*p);
  g->build();
  g->make_window(p->window_requests);
  return g;
}

void ws_next_window(void* h, uint32_t R) { static_cast<Gen*>(h)->make_window(R); }

// sizes: [I, R, window chain blocks, seed chains, seed blocks]
void ws_sizes(void* h, uint64_t* out) {
  Gen* g = static_cast<Gen*>(h);
  out[0] = g->p.num_instances;
  out[1] = g->w_len.size();
  out[2] = g->w_hash.size();
  out[3] = g->c_inst.size();
  out[4] = g->c_hash.size();
}

void ws_copy_window(void* h, uint64_t* off, uint64_t* hash, uint32_t* len, float* ttft, float* tpot,
                    uint32_t* session, uint32_t* out_tokens) {
  Gen* g = static_cast<Gen*>(h);
  std::memcpy(off, g->w_off.data(), g->w_off.size() * 8);
  if (!g->w_hash.empty()) std::memcpy(hash, g->w_hash.data(), g->w_hash.size() * 8);
  size_t R = g->w_len.size();
  if (R) {
    std::memcpy(len, g->w_len.data(), R * 4);
    std::memcpy(ttft, g->w_ttft.data(), R * 4);
    std::memcpy(tpot, g->w_tpot.data(), R * 4);
    std::memcpy(session, g->w_sess.data(), R * 4);
    std::memcpy(out_tokens, g->w_out.data(), R * 4);
  }
}

void ws_copy_instances(void* h, int32_t* b, int32_t* qr, int64_t* q, int64_t* S, int64_t* M,
                       int32_t* bmax, uint64_t* cap) {
  Gen* g = static_cast<Gen*>(h);
  size_t I = g->p.num_instances;
  std::memcpy(b, g->s_b.data(), I * 4);
  std::memcpy(qr, g->s_qr.data(), I * 4);
  std::memcpy(q, g->s_q.data(), I * 8);
  std::memcpy(S, g->s_S.data(), I * 8);
  std::memcpy(M, g->s_M.data(), I * 8);
  std::memcpy(bmax, g->s_bmax.data(), I * 4);
  std::memcpy(cap, g->s_cap.data(), I * 8);
}

void ws_copy_seed_chains(void* h, uint32_t* inst, uint64_t* off, uint64_t* hash, uint64_t* parent) {
  Gen* g = static_cast<Gen*>(h);
  size_t n = g->c_inst.size();
  if (n) {
    std::memcpy(inst, g->c_inst.data(), n * 4);
    std::memcpy(parent, g->c_parent.data(), n * 8);
  }
  std::memcpy(off, g->c_off.data(), (n + 1) * 8);
  if (!g->c_hash.empty()) std::memcpy(hash, g->c_hash.data(), g->c_hash.size() * 8);
}

// Requests in flight at the start of a stream, consistent with the instance state's counts: per
// instance, b decoding requests (prompt U{1024..16384} tokens, output U{16..1024}, remaining output
// U{1..output}) and qr queued ones holding the queued prefill tokens q in FIFO chunks of 4096 (the
// remainder last), each with a prompt of its chunk plus U{0..8192} cached tokens.  With inst == NULL
// only the count is returned.
uint64_t ws_initial_requests(void* h, uint32_t* inst, uint32_t* state, uint32_t* L, uint32_t* out,
                             uint64_t* rem) {
  Gen* g = static_cast<Gen*>(h);
  uint64_t n = 0;
  for (uint32_t i = 0; i < g->p.num_instances; ++i) {
    Rng rr(g->p.seed, kPurposeRequests, i);
    for (int32_t k = 0; k < g->s_b[i]; ++k, ++n) {
      const uint32_t l = (uint32_t)rr.range(1024, 16384);
      const uint32_t o = (uint32_t)rr.range(16, 1024);
      const uint32_t left = (uint32_t)rr.range(1, o);
      if (inst) { inst[n] = i; state[n] = 1; L[n] = l; out[n] = o; rem[n] = left; }
    }
    int64_t q = g->s_q[i];
    for (int32_t k = 0; k < g->s_qr[i]; ++k, ++n) {
      const int64_t chunk = k + 1 < g->s_qr[i] ? 4096 : q;
      q -= chunk;
      const uint32_t l = (uint32_t)(chunk + rr.range(0, 8192));
      const uint32_t o = (uint32_t)rr.range(16, 1024);
      if (inst) { inst[n] = i; state[n] = 0; L[n] = l; out[n] = o; rem[n] = (uint64_t)chunk; }
    }
  }
  return n;
}

// Drop the instance seed chains (they can be large) once the caller has copied them.
void ws_release_seed_chains(void* h) {
  Gen* g = static_cast<Gen*>(h);
  std::vector<uint32_t>().swap(g->c_inst);
  std::vector<uint64_t>().swap(g->c_hash);
  std::vector<uint64_t>().swap(g->c_parent);
  g->c_off.assign(1, 0);
}

void ws_free(void* h) { delete static_cast<Gen*>(h); }

// Block-hash chain of an explicit token list (full blocks only): the same chaining as above.
uint64_t ws_chain_from_tokens(const uint32_t* tokens, uint64_t n_tokens, uint64_t* out) {
  uint64_t nblk = n_tokens / 16, x = 0;
  for (uint64_t k = 0; k < nblk; ++k) {
    for (uint64_t j = 0; j < 16; ++j) x = splitmix64(x ^ (uint64_t)tokens[16 * k + j]);
    if (x == 0) x = 1;
    out[k] = x;
  }
  return nblk;
}

// Test hooks for the deterministic series (compared against libm in the generator's own tests).
double ws_det_exp(double x) { return det_exp(x); }
double ws_det_log(double x) { return det_log(x); }

}  // extern "C"
