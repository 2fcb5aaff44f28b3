// Host implementation of the C ABI declared in include/packserve.h.
//
// Owns every device allocation (made in ps_create), validates arguments on the host (or with a
// device-side check kernel when the caller passes device buffers), orders all work on one stream,
// and turns the device error word into a ps_status at the end of each call.
#include <cmath>
#include <cstdio>
#include <cstring>
#include <string>
#include <vector>

#include <algorithm>

#include "packserve.h"
#include "calibrate.h"
#include "ps_internal.cuh"

namespace {

// Events on the context's stream: four timed phases (start/end pairs), then the two split points of
// the probe phase (after the relations kernel, between the two probe kernels).
enum Ev { kEvProbe0, kEvProbe1, kEvScore0, kEvScore1, kEvGreedy0, kEvGreedy1, kEvCommit0, kEvCommit1, kEvRelDone,
          kEvProbeMid, kNumEv };
constexpr int kNumPhases = 4;
constexpr int kNumStats = 6;
constexpr uint64_t kDefaultWaitNs = 1000000000ull;  // 1 s: bound on a cross-block wait of the greedy

struct DeviceGuard {
  int prev = -1;
  explicit DeviceGuard(int dev) {
    if (cudaGetDevice(&prev) != cudaSuccess) prev = -1;
    if (prev != dev) cudaSetDevice(dev);
  }
  ~DeviceGuard() {
    int cur = -1;
    if (prev >= 0 && cudaGetDevice(&cur) == cudaSuccess && cur != prev) cudaSetDevice(prev);
  }
};

}  // namespace

struct ps_ctx {
  int device = 0;
  cudaStream_t stream = nullptr;
  bool own_stream = false;
  uint32_t I = 0, Rmax = 0;
  uint64_t max_blocks = 0;
  psk::DevModel model{};
  int num_sms = 0, probe_grid = 0;
  int search = 0;  // PS_PROBE_SEARCH
  std::vector<uint64_t> cap;
  uint64_t total_slots = 0;
  uint64_t* d_slots = nullptr;
  uint64_t total_ovf = 0;
  uint64_t* d_ovf = nullptr;
  psk::TableDesc* d_tdesc = nullptr;
  unsigned long long* d_count = nullptr;
  psk::DeltaSlot* d_delta = nullptr;
  uint64_t delta_nslots = 0;
  psk::GreedySync gsync{nullptr, nullptr, nullptr, nullptr, nullptr, 0u, kDefaultWaitNs, nullptr, nullptr, nullptr};
  psk::RowPre* d_rows = nullptr;      // per-request constants and relations (search mode greedy)
  psk::LastSlot* d_lastslot = nullptr;
  psk::RowList scratch{nullptr, nullptr};  // rows the probe searches from scratch
  uint32_t lastslot_n = 0;
  psk::StateSoA st{}, pend{};
  uint64_t* d_off = nullptr;
  uint64_t* d_hash = nullptr;
  // shared-prefix windows (ps_window.parent): each request's own blocks and parent link, staged
  uint64_t* d_own_off = nullptr;
  uint64_t* d_own_hash = nullptr;
  int32_t* d_parent = nullptr;
  std::vector<uint64_t> h_full_off;
  uint32_t* d_L = nullptr;
  float* d_ttft = nullptr;
  float* d_tpot = nullptr;
  uint32_t* d_hits = nullptr;
  float* d_tpf = nullptr;  // T_pf at each pair's hit, from the probe, for the greedy pass
  float* d_tpot_o = nullptr;
  float* d_ttft_o = nullptr;
  uint8_t* d_cls = nullptr;
  int32_t* d_best = nullptr;
  uint8_t* d_path = nullptr;
  int32_t* d_assign = nullptr;
  uint8_t* d_dpath = nullptr;
  uint32_t* d_hchosen = nullptr;
  uint32_t* d_err = nullptr;
  uint32_t* h_err = nullptr;   // pinned: the device error word, read at the end of each call
  uint32_t* h_more = nullptr;  // pinned: "another eviction round" flag
  cudaEvent_t ev[kNumEv] = {};
  bool ev_used[kNumPhases] = {};
  bool probe_split = false;            // kEvRelDone / kEvProbeMid recorded in the last probe phase
  unsigned long long* d_stats = nullptr;  // probe launch counters (ps_last_probe_stats)
  bool pending = false;
  psk::WindowDev pend_win{};
  // column-block scoring: the window of the last ps_shard_wmin, whose hits are in d_hits
  bool shard_pending = false;
  psk::WindowDev shard_win{};
  uint32_t* d_shard_wmin = nullptr;
  unsigned long long* d_shard_key = nullptr;
  uint32_t* d_shard_tie = nullptr;
  const uint32_t* pend_out = nullptr;
  // streaming: per-block LRU metadata, request store, capacities on the device, eviction buffers
  bool lru = false;
  psk::LruMeta meta{nullptr, nullptr, nullptr};
  void* d_leafbuf = nullptr;
  unsigned long long* d_cprefix = nullptr;  // [2 (Rmax + 1)] commit item prefixes
  uint32_t* d_nleaf = nullptr;
  uint32_t* d_more = nullptr;
  uint64_t max_instance_slots = 0;
  psk::ReqStore rq{};
  uint64_t* d_cap = nullptr;
  uint32_t* d_outtok = nullptr;
  std::vector<void*> allocs;
  std::string err;
};

namespace {

ps_status fail(ps_ctx* c, ps_status s, const std::string& msg) {
  if (c) c->err = msg;
  return s;
}

#define PS_TRY_CUDA(ctx, call)                                                                     \
  do {                                                                                             \
    cudaError_t e_ = (call);                                                                       \
    if (e_ != cudaSuccess)                                                                         \
      return fail((ctx), PS_ERR_CUDA, std::string(#call) + ": " + cudaGetErrorString(e_));         \
  } while (0)

template <class T>
cudaError_t dalloc(ps_ctx* c, T** p, size_t count) {
  void* v = nullptr;
  const size_t bytes = count ? count * sizeof(T) : sizeof(T);
  cudaError_t e = cudaMalloc(&v, bytes);
  if (e != cudaSuccess) return e;
  c->allocs.push_back(v);
  *p = static_cast<T*>(v);
  return cudaSuccess;
}

bool finite_small(float x) { return std::isfinite(x) && std::fabs(x) <= 1e9f; }

ps_status check_model(ps_ctx* c, const ps_model& m) {
  const float coeffs[] = {m.a0, m.a1, m.a2, m.a3, m.a4, m.a5, m.b0, m.b1, m.b2, m.g_q, m.eta, m.lout_median};
  for (float x : coeffs)
    if (!finite_small(x)) return fail(c, PS_ERR_INVALID, "model coefficient not finite or |x| > 1e9");
  if (m.eta < 0.0f) return fail(c, PS_ERR_INVALID, "eta must be >= 0 (Eq. 8)");
  if (m.interference_mode != 0 && m.interference_mode != 1)
    return fail(c, PS_ERR_INVALID, "interference_mode must be 0 or 1");
  if (m.ttft_filter != 0 && m.ttft_filter != 1) return fail(c, PS_ERR_INVALID, "ttft_filter must be 0 or 1");
  if (m.nseg < 1 || m.nseg > PS_MAX_EMA_SEGMENTS) return fail(c, PS_ERR_INVALID, "nseg must be 1..16");
  for (int s = 0; s < m.nseg; ++s) {
    if (!(std::isfinite(m.ema_factor[s]) && m.ema_factor[s] > 0.0f && m.ema_factor[s] <= 1e9f))
      return fail(c, PS_ERR_INVALID, "EMA factors must be finite and > 0");
    if (s > 0 && m.seg_lo[s] <= m.seg_lo[s - 1]) return fail(c, PS_ERR_INVALID, "seg_lo must ascend");
  }
  if (m.seg_lo[0] > 1) return fail(c, PS_ERR_INVALID, "seg_lo[0] must be <= 1");
  if ((m.cache_filter_off | m.slo_filter_off | m.fallback_dcq) & ~1)
    return fail(c, PS_ERR_INVALID, "cache_filter_off, slo_filter_off and fallback_dcq must be 0 or 1");
  if (m.selector < PS_SELECT_DCQ || m.selector > PS_SELECT_HCQ) return fail(c, PS_ERR_INVALID, "selector must be 0..5");
  return PS_OK;
}

psk::DevModel to_dev(const ps_model& m) {
  psk::DevModel d{};
  d.a0 = m.a0; d.a1 = m.a1; d.a2 = m.a2; d.a3 = m.a3; d.a4 = m.a4; d.a5 = m.a5;
  d.b0 = m.b0; d.b1 = m.b1; d.b2 = m.b2; d.g_q = m.g_q; d.eta = m.eta; d.lout = m.lout_median;
  d.interference_mode = m.interference_mode;
  d.ttft_filter = m.ttft_filter;
  d.nseg = m.nseg;
  for (int s = 0; s < PS_MAX_EMA_SEGMENTS; ++s) {
    d.seg_lo[s] = m.seg_lo[s];
    d.ema[s] = m.ema_factor[s];
  }
  d.cache_off = m.cache_filter_off;
  d.slo_off = m.slo_filter_off;
  d.fb_dcq = m.fallback_dcq;
  d.sel = m.selector;
  return d;
}

ps_status device_errors(ps_ctx* c) {
  const uint32_t e = *c->h_err;
  if (e == 0) return PS_OK;
  if (e & psk::kErrWindowLayout)
    return fail(c, PS_ERR_INVALID, "window layout: chain_off must start at 0, ascend, give L/16 blocks per "
                                   "request, L < 2^30, and stay within max_window_chain_blocks");
  if (e & psk::kErrBadInstance) return fail(c, PS_ERR_INVALID, "instance id out of range");
  if (e & psk::kErrReservedHash) return fail(c, PS_ERR_INVALID, "block hash 0 or 2^64-1 is reserved");
  if (e & psk::kErrParentMissing)
    return fail(c, PS_ERR_INVALID, "a chain's parent_hash is not cached (PS_PROBE_SEARCH needs prefix-closed caches)");
  if (e & psk::kErrDeltaFull) return fail(c, PS_ERR_TABLE_FULL, "window delta table full");
  if (e & psk::kErrTimeout) return fail(c, PS_ERR_TIMEOUT, "a bounded device-side wait gave up");
  if (e & psk::kErrRequestsFull)
    return fail(c, PS_ERR_CAPACITY, "an instance has more requests in flight than max_active_requests");
  if (e & psk::kErrLeavesFull)
    return fail(c, PS_ERR_TABLE_FULL, "an instance has more leaf blocks than the eviction buffer (4096)");
  if (e & psk::kErrTableFull) return fail(c, PS_ERR_TABLE_FULL, "instance hash table full");
  return fail(c, PS_ERR_CUDA, "unknown device error");
}

// Synchronise the stream, read the device error word, and reset it for the next call.
ps_status finish(ps_ctx* c) {
  PS_TRY_CUDA(c, cudaMemcpyAsync(c->h_err, c->d_err, sizeof(uint32_t), cudaMemcpyDeviceToHost, c->stream));
  PS_TRY_CUDA(c, cudaStreamSynchronize(c->stream));
  ps_status s = device_errors(c);
  if (*c->h_err) {
    PS_TRY_CUDA(c, cudaMemsetAsync(c->d_err, 0, sizeof(uint32_t), c->stream));
    PS_TRY_CUDA(c, cudaStreamSynchronize(c->stream));
    *c->h_err = 0;
  }
  return s;
}

ps_status check_capacity(ps_ctx* c) {
  std::vector<unsigned long long> cnt(c->I);
  PS_TRY_CUDA(c, cudaMemcpy(cnt.data(), c->d_count, c->I * sizeof(unsigned long long), cudaMemcpyDeviceToHost));
  for (uint32_t i = 0; i < c->I; ++i)
    if (cnt[i] > c->cap[i])
      return fail(c, PS_ERR_CAPACITY, "instance " + std::to_string(i) + " holds " + std::to_string(cnt[i]) +
                                          " blocks > capacity " + std::to_string(c->cap[i]));
  return PS_OK;
}

// Copies the request arrays shared by both window forms (L, targets, output lengths) to the device.
ps_status stage_request_arrays(ps_ctx* c, const ps_window* w) {
  if (!w->R) return PS_OK;
  PS_TRY_CUDA(c, cudaMemcpyAsync(c->d_L, w->prompt_tokens, w->R * sizeof(uint32_t), cudaMemcpyHostToDevice, c->stream));
  PS_TRY_CUDA(c, cudaMemcpyAsync(c->d_ttft, w->ttft_target, w->R * sizeof(float), cudaMemcpyHostToDevice, c->stream));
  PS_TRY_CUDA(c, cudaMemcpyAsync(c->d_tpot, w->tpot_target, w->R * sizeof(float), cudaMemcpyHostToDevice, c->stream));
  if (w->out_tokens) {
    PS_TRY_CUDA(c, cudaMemcpyAsync(c->d_outtok, w->out_tokens, w->R * sizeof(uint32_t), cudaMemcpyHostToDevice,
                                   c->stream));
    c->pend_out = c->d_outtok;
  }
  return PS_OK;
}

// Shared-prefix form (host inputs): validate the parent links and own-block counts, send each
// request's own blocks, and rebuild the full chains on the device.
ps_status stage_window_tree(ps_ctx* c, const ps_window* w, psk::WindowDev* out) {
  const uint32_t R = w->R;
  const uint64_t* own = w->chain_off;
  if (own[0] != 0) return fail(c, PS_ERR_INVALID, "chain_off[0] must be 0");
  std::vector<uint64_t>& full = c->h_full_off;
  full.assign((size_t)R + 1, 0);
  for (uint32_t r = 0; r < R; ++r) {
    const uint32_t L = w->prompt_tokens[r];
    const int32_t p = w->parent[r];
    if (L >= (1u << 30)) return fail(c, PS_ERR_INVALID, "request " + std::to_string(r) + ": L must be < 2^30");
    if (p < -1 || p >= (int64_t)r)
      return fail(c, PS_ERR_INVALID, "request " + std::to_string(r) + ": parent must be -1 or an earlier request");
    const uint64_t nb = L / 16u;
    const uint64_t pb = p >= 0 ? full[(size_t)p + 1] - full[(size_t)p] : 0;
    if (own[r + 1] < own[r] || nb < pb || own[r + 1] - own[r] != nb - pb)
      return fail(c, PS_ERR_INVALID, "request " + std::to_string(r) +
                                         ": own blocks must be L/16 minus the parent's chain length");
    full[(size_t)r + 1] = full[r] + nb;
  }
  const uint64_t nblk = full[R], nown = own[R];
  if (nblk > c->max_blocks) return fail(c, PS_ERR_INVALID, "window exceeds max_window_chain_blocks");
  if (nown > 0 && !w->chain_hash) return fail(c, PS_ERR_INVALID, "chain_hash is NULL");
  PS_TRY_CUDA(c, cudaMemcpyAsync(c->d_off, full.data(), ((size_t)R + 1) * sizeof(uint64_t), cudaMemcpyHostToDevice,
                                 c->stream));
  if (R) {
    PS_TRY_CUDA(c, cudaMemcpyAsync(c->d_own_off, own, ((size_t)R + 1) * sizeof(uint64_t), cudaMemcpyHostToDevice,
                                   c->stream));
    PS_TRY_CUDA(c, cudaMemcpyAsync(c->d_parent, w->parent, R * sizeof(int32_t), cudaMemcpyHostToDevice, c->stream));
  }
  if (nown)
    PS_TRY_CUDA(c, cudaMemcpyAsync(c->d_own_hash, w->chain_hash, nown * sizeof(uint64_t), cudaMemcpyHostToDevice,
                                   c->stream));
  ps_status s = stage_request_arrays(c, w);
  if (s != PS_OK) return s;
  PS_TRY_CUDA(c, pskl::launch_expand_chains(c->d_off, c->d_own_off, c->d_own_hash, c->d_parent, R, c->d_hash, c->d_err,
                                            c->num_sms, c->stream));
  out->off = c->d_off;
  out->hash = c->d_hash;
  out->L = c->d_L;
  out->ttft_t = c->d_ttft;
  out->tpot_t = c->d_tpot;
  return PS_OK;
}

// Validate a window and make its arrays available on the device.
ps_status stage_window(ps_ctx* c, const ps_window* w, psk::WindowDev* out) {
  if (!w) return fail(c, PS_ERR_INVALID, "window is NULL");
  if (w->R > c->Rmax) return fail(c, PS_ERR_INVALID, "window has more than max_window_requests requests");
  if (w->inputs_on_device != 0 && w->inputs_on_device != 1)
    return fail(c, PS_ERR_INVALID, "inputs_on_device must be 0 or 1");
  if (!w->chain_off || (w->R > 0 && (!w->prompt_tokens || !w->ttft_target || !w->tpot_target)))
    return fail(c, PS_ERR_INVALID, "window array is NULL");
  out->R = w->R;
  c->pend_out = nullptr;
  if (w->inputs_on_device) {
    if (w->parent) return fail(c, PS_ERR_INVALID, "a window with parent links must be in host memory");
    c->pend_out = w->out_tokens;
    out->off = w->chain_off;
    out->hash = w->chain_hash;
    out->L = w->prompt_tokens;
    out->ttft_t = w->ttft_target;
    out->tpot_t = w->tpot_target;
    if (w->R > 0) {
      PS_TRY_CUDA(c, pskl::launch_validate_window(*out, c->max_blocks, c->d_err, c->stream));
      ps_status s = finish(c);
      if (s != PS_OK) return s;
      uint64_t nblk = 0;
      PS_TRY_CUDA(c, cudaMemcpy(&nblk, w->chain_off + w->R, sizeof(uint64_t), cudaMemcpyDeviceToHost));
      if (nblk > 0 && !w->chain_hash) return fail(c, PS_ERR_INVALID, "chain_hash is NULL");
    }
    return PS_OK;
  }
  if (w->parent) return stage_window_tree(c, w, out);
  const uint64_t* off = w->chain_off;
  if (off[0] != 0) return fail(c, PS_ERR_INVALID, "chain_off[0] must be 0");
  for (uint32_t r = 0; r < w->R; ++r) {
    const uint32_t L = w->prompt_tokens[r];
    if (off[r + 1] < off[r] || off[r + 1] - off[r] != (uint64_t)(L / 16u) || L >= (1u << 30))
      return fail(c, PS_ERR_INVALID, "request " + std::to_string(r) + ": chain length must be L/16 blocks, L < 2^30");
  }
  const uint64_t nblk = off[w->R];
  if (nblk > c->max_blocks) return fail(c, PS_ERR_INVALID, "window exceeds max_window_chain_blocks");
  if (nblk > 0 && !w->chain_hash) return fail(c, PS_ERR_INVALID, "chain_hash is NULL");
  PS_TRY_CUDA(c, cudaMemcpyAsync(c->d_off, off, (w->R + 1) * sizeof(uint64_t), cudaMemcpyHostToDevice, c->stream));
  if (nblk)
    PS_TRY_CUDA(c, cudaMemcpyAsync(c->d_hash, w->chain_hash, nblk * sizeof(uint64_t), cudaMemcpyHostToDevice, c->stream));
  ps_status s = stage_request_arrays(c, w);
  if (s != PS_OK) return s;
  out->off = c->d_off;
  out->hash = c->d_hash;
  out->L = c->d_L;
  out->ttft_t = c->d_ttft;
  out->tpot_t = c->d_tpot;
  return PS_OK;
}

// Copy n elements of scratch to a caller buffer (host or device).
template <class T>
cudaError_t deliver(ps_ctx* c, T* dst, const T* src, size_t n, int on_device) {
  if (!dst || n == 0 || dst == src) return cudaSuccess;
  return cudaMemcpyAsync(dst, src, n * sizeof(T), on_device ? cudaMemcpyDeviceToDevice : cudaMemcpyDeviceToHost,
                         c->stream);
}

void record(ps_ctx* c, int ev) { cudaEventRecord(c->ev[ev], c->stream); }

ps_status run_probe_and_score(ps_ctx* c, const psk::WindowDev& wd, ps_scores* out, uint32_t** hits_used) {
  const int dev_out = out ? out->outputs_on_device : 0;
  uint32_t* hits = (out && out->hits && dev_out) ? out->hits : c->d_hits;
  PS_TRY_CUDA(c, cudaMemsetAsync(c->d_stats, 0, kNumStats * sizeof(unsigned long long), c->stream));
  record(c, kEvProbe0);
  // window relations first: the probe derives the rows of requests that extend an earlier request
  PS_TRY_CUDA(c, pskl::launch_relations(wd, c->model, c->d_lastslot, c->lastslot_n, c->d_rows, c->scratch, c->num_sms,
                                        c->stream));
  record(c, kEvRelDone);
  PS_TRY_CUDA(c, pskl::launch_probe(c->d_slots, c->d_ovf, c->d_tdesc, c->I, wd, c->d_rows, c->scratch, hits, c->d_tpf,
                                    c->model, c->probe_grid, c->search, c->d_stats, c->ev[kEvProbeMid], c->stream));
  record(c, kEvProbe1);
  c->ev_used[0] = true;
  c->probe_split = wd.R > 0;
  *hits_used = hits;
  if (!out) return PS_OK;
  const size_t RI = (size_t)wd.R * c->I;
  const bool want_score = out->tpot || out->ttft || out->cls || out->best || out->path;
  if (want_score) {
    float* tpot = out->tpot ? (dev_out ? out->tpot : c->d_tpot_o) : nullptr;
    float* ttft = out->ttft ? (dev_out ? out->ttft : c->d_ttft_o) : nullptr;
    uint8_t* cls = out->cls ? (dev_out ? out->cls : c->d_cls) : nullptr;
    int32_t* best = out->best ? (dev_out ? out->best : c->d_best) : nullptr;
    uint8_t* path = out->path ? (dev_out ? out->path : c->d_path) : nullptr;
    record(c, kEvScore0);
    PS_TRY_CUDA(c, pskl::launch_score(hits, c->st, c->I, wd, c->model, tpot, ttft, cls, best, path, c->num_sms,
                                      c->stream));
    record(c, kEvScore1);
    c->ev_used[1] = true;
    if (!dev_out) {
      PS_TRY_CUDA(c, deliver(c, out->tpot, c->d_tpot_o, RI, 0));
      PS_TRY_CUDA(c, deliver(c, out->ttft, c->d_ttft_o, RI, 0));
      PS_TRY_CUDA(c, deliver(c, out->cls, c->d_cls, RI, 0));
      PS_TRY_CUDA(c, deliver(c, out->best, c->d_best, wd.R, 0));
      PS_TRY_CUDA(c, deliver(c, out->path, c->d_path, wd.R, 0));
    }
  }
  if (out->hits && !dev_out) PS_TRY_CUDA(c, deliver(c, out->hits, c->d_hits, RI, 0));
  return PS_OK;
}

void reset_timers(ps_ctx* c) {
  for (bool& u : c->ev_used) u = false;
  c->probe_split = false;
  c->shard_pending = false;  // the hit buffer is about to be rewritten
}

}  // namespace

extern "C" {

ps_status ps_create(const ps_config* cfg, ps_ctx** out) {
  if (!out) return PS_ERR_INVALID;
  *out = nullptr;
  if (!cfg) return PS_ERR_INVALID;
  ps_ctx* c = new ps_ctx();
  auto bail = [&](ps_status s) {
    ps_destroy(c);
    return s;
  };
  if (cfg->num_instances < 1 || cfg->num_instances > 2048) return bail(PS_ERR_INVALID);
  if (cfg->max_window_requests < 1 || cfg->max_window_requests > (1u << 17)) return bail(PS_ERR_INVALID);
  if (cfg->max_window_chain_blocks < 1 || cfg->max_window_chain_blocks > (1ull << 36)) return bail(PS_ERR_INVALID);
  if (cfg->block_tokens != PS_BLOCK_TOKENS || !cfg->cap_blocks) return bail(PS_ERR_INVALID);
  if (!(cfg->table_load_factor > 0.0f && cfg->table_load_factor <= 0.95f)) return bail(PS_ERR_INVALID);
  if (check_model(c, cfg->model) != PS_OK) return bail(PS_ERR_INVALID);
  if (cfg->probe_mode != PS_PROBE_LINEAR && cfg->probe_mode != PS_PROBE_SEARCH) return bail(PS_ERR_INVALID);
  c->search = cfg->probe_mode == PS_PROBE_SEARCH ? 1 : 0;
  if (cfg->track_lru != 0 && cfg->track_lru != 1) return bail(PS_ERR_INVALID);
  if (cfg->max_active_requests > (1u << 16)) return bail(PS_ERR_INVALID);
  c->lru = cfg->track_lru == 1;
  c->rq.M = cfg->max_active_requests;
  c->device = cfg->device;
  c->I = cfg->num_instances;
  c->Rmax = cfg->max_window_requests;
  c->max_blocks = cfg->max_window_chain_blocks;
  c->model = to_dev(cfg->model);
  c->cap.assign(cfg->cap_blocks, cfg->cap_blocks + c->I);
  DeviceGuard g(c->device);
  if (cudaSetDevice(c->device) != cudaSuccess) return bail(PS_ERR_CUDA);
  if (cudaDeviceGetAttribute(&c->num_sms, cudaDevAttrMultiProcessorCount, c->device) != cudaSuccess)
    return bail(PS_ERR_CUDA);
  if (cfg->cuda_stream) {
    c->stream = static_cast<cudaStream_t>(cfg->cuda_stream);
  } else {
    if (cudaStreamCreateWithFlags(&c->stream, cudaStreamNonBlocking) != cudaSuccess) return bail(PS_ERR_CUDA);
    c->own_stream = true;
  }
  // Instance tables: slots = ceil(cap / lf) rounded up to whole 8-slot buckets; one overflow bit
  // per bucket, each instance's bitmap starting on its own u64 word.
  std::vector<psk::TableDesc> td(c->I);
  uint64_t base = 0, obase = 0;
  for (uint32_t i = 0; i < c->I; ++i) {
    if (c->cap[i] < 1 || c->cap[i] > (1ull << 36)) return bail(PS_ERR_INVALID);
    const uint64_t slots = (uint64_t)std::ceil((double)c->cap[i] / (double)cfg->table_load_factor);
    const uint64_t nbkt = (slots + psk::kBucketSlots - 1) / psk::kBucketSlots;
    if (nbkt >= (1ull << 32)) return bail(PS_ERR_INVALID);
    td[i].base = base;
    td[i].ovf = obase;
    td[i].nbkt = (uint32_t)nbkt;
    td[i].pad = 0;
    base += nbkt * psk::kBucketSlots;
    obase += (nbkt + 63) / 64;
  }
  c->total_slots = base;
  if (c->lru && c->total_slots >= (1ull << 32) - 2) {
    c->err = "track_lru needs fewer than 2^32 - 2 table slots in total (eviction keeps 32-bit slot indices)";
    return bail(PS_ERR_INVALID);
  }
  c->total_ovf = obase;
  const uint64_t dn = std::max<uint64_t>(16, 2 * c->max_blocks);  // delta slots: twice a window's blocks
  c->delta_nslots = dn;
  c->lastslot_n = 64;
  while (c->lastslot_n < 2 * c->Rmax) c->lastslot_n <<= 1;
  const size_t RI = (size_t)c->Rmax * c->I;
  const size_t I = c->I;
  c->gsync.ring_stride = (c->I + 3u) / 4u * 4u;
  bool ok = dalloc(c, &c->d_slots, c->total_slots) == cudaSuccess && dalloc(c, &c->d_ovf, c->total_ovf) == cudaSuccess &&
            dalloc(c, &c->d_tdesc, I) == cudaSuccess && dalloc(c, &c->d_count, I) == cudaSuccess &&
            dalloc(c, &c->d_delta, (size_t)dn) == cudaSuccess && dalloc(c, &c->gsync.jobs, c->Rmax) == cudaSuccess &&
            dalloc(c, &c->gsync.done, c->Rmax) == cudaSuccess && dalloc(c, &c->gsync.ready, c->Rmax) == cudaSuccess &&
            dalloc(c, &c->gsync.sums, psk::kSumSlots) == cudaSuccess && dalloc(c, &c->gsync.sready, c->Rmax) == cudaSuccess &&
            dalloc(c, &c->gsync.stats, psk::kGreedyStats) == cudaSuccess &&
            dalloc(c, &c->gsync.hitring, (size_t)psk::kHitSlots * c->gsync.ring_stride) == cudaSuccess &&
            dalloc(c, &c->gsync.tpfring, (size_t)psk::kHitSlots * c->gsync.ring_stride) == cudaSuccess &&
            dalloc(c, &c->d_rows, c->Rmax) == cudaSuccess && dalloc(c, &c->d_lastslot, c->lastslot_n) == cudaSuccess &&
            dalloc(c, &c->scratch.rows, c->Rmax) == cudaSuccess && dalloc(c, &c->scratch.count, 1) == cudaSuccess &&
            dalloc(c, &c->d_cprefix, 2 * ((size_t)c->Rmax + 1)) == cudaSuccess;
  for (psk::StateSoA* s : {&c->st, &c->pend}) {
    ok = ok && dalloc(c, &s->b, I) == cudaSuccess && dalloc(c, &s->qr, I) == cudaSuccess &&
         dalloc(c, &s->q, I) == cudaSuccess && dalloc(c, &s->S, I) == cudaSuccess &&
         dalloc(c, &s->M, I) == cudaSuccess && dalloc(c, &s->Bmax, I) == cudaSuccess;
  }
  ok = ok && dalloc(c, &c->d_off, (size_t)c->Rmax + 1) == cudaSuccess &&
       dalloc(c, &c->d_hash, c->max_blocks) == cudaSuccess &&
       dalloc(c, &c->d_own_off, (size_t)c->Rmax + 1) == cudaSuccess &&
       dalloc(c, &c->d_own_hash, c->max_blocks) == cudaSuccess && dalloc(c, &c->d_parent, c->Rmax) == cudaSuccess && dalloc(c, &c->d_L, c->Rmax) == cudaSuccess &&
       dalloc(c, &c->d_ttft, c->Rmax) == cudaSuccess && dalloc(c, &c->d_tpot, c->Rmax) == cudaSuccess &&
       dalloc(c, &c->d_hits, RI) == cudaSuccess && dalloc(c, &c->d_tpf, RI) == cudaSuccess && dalloc(c, &c->d_tpot_o, RI) == cudaSuccess &&
       dalloc(c, &c->d_ttft_o, RI) == cudaSuccess && dalloc(c, &c->d_cls, RI) == cudaSuccess &&
       dalloc(c, &c->d_best, c->Rmax) == cudaSuccess && dalloc(c, &c->d_path, c->Rmax) == cudaSuccess &&
       dalloc(c, &c->d_assign, c->Rmax) == cudaSuccess && dalloc(c, &c->d_dpath, c->Rmax) == cudaSuccess &&
       dalloc(c, &c->d_hchosen, c->Rmax) == cudaSuccess && dalloc(c, &c->d_err, 1) == cudaSuccess &&
       dalloc(c, &c->d_stats, kNumStats) == cudaSuccess && dalloc(c, &c->d_shard_wmin, c->Rmax) == cudaSuccess &&
       dalloc(c, &c->d_shard_key, c->Rmax) == cudaSuccess && dalloc(c, &c->d_shard_tie, c->Rmax) == cudaSuccess &&
       dalloc(c, &c->d_cap, I) == cudaSuccess && dalloc(c, &c->d_outtok, c->Rmax) == cudaSuccess;
  if (ok && c->lru) {
    for (uint32_t i = 0; i < I; ++i)
      c->max_instance_slots = std::max<uint64_t>(c->max_instance_slots, (uint64_t)td[i].nbkt * psk::kBucketSlots);
    unsigned char* lb = nullptr;
    ok = dalloc(c, &lb, pskl::evict_leafbuf_bytes(c->I)) == cudaSuccess && dalloc(c, &c->d_nleaf, I) == cudaSuccess &&
         dalloc(c, &c->d_more, 1) == cudaSuccess;
    c->d_leafbuf = lb;
  }
  if (ok && c->lru)
    ok = dalloc(c, &c->meta.last_use, c->total_slots) == cudaSuccess &&
         dalloc(c, &c->meta.children, c->total_slots) == cudaSuccess &&
         dalloc(c, &c->meta.parent, c->total_slots) == cudaSuccess;
  if (ok && c->rq.M) {
    const size_t IM = I * (size_t)c->rq.M;
    ok = dalloc(c, &c->rq.q_head, I) == cudaSuccess && dalloc(c, &c->rq.q_len, I) == cudaSuccess &&
         dalloc(c, &c->rq.q_L, IM) == cudaSuccess && dalloc(c, &c->rq.q_out, IM) == cudaSuccess &&
         dalloc(c, &c->rq.q_rem, IM) == cudaSuccess && dalloc(c, &c->rq.d_len, I) == cudaSuccess &&
         dalloc(c, &c->rq.d_L, IM) == cudaSuccess && dalloc(c, &c->rq.d_out, IM) == cudaSuccess &&
         dalloc(c, &c->rq.d_rem, IM) == cudaSuccess;
  }
  if (!ok) {
    cudaGetLastError();
    return bail(PS_ERR_OOM);
  }
  if (cudaMallocHost(&c->h_err, sizeof(uint32_t)) != cudaSuccess) return bail(PS_ERR_OOM);
  *c->h_err = 0;
  if (cudaMallocHost(&c->h_more, sizeof(uint32_t)) != cudaSuccess) return bail(PS_ERR_OOM);
  *c->h_more = 0;
  for (int e = 0; e < kNumEv; ++e)
    if (cudaEventCreate(&c->ev[e]) != cudaSuccess) return bail(PS_ERR_CUDA);
  bool set = cudaMemsetAsync(c->d_slots, 0, c->total_slots * sizeof(uint64_t), c->stream) == cudaSuccess &&
             cudaMemsetAsync(c->d_ovf, 0, c->total_ovf * sizeof(uint64_t), c->stream) == cudaSuccess &&
             cudaMemcpyAsync(c->d_tdesc, td.data(), I * sizeof(psk::TableDesc), cudaMemcpyHostToDevice,
                             c->stream) == cudaSuccess &&
             cudaMemsetAsync(c->d_count, 0, I * sizeof(unsigned long long), c->stream) == cudaSuccess &&
             cudaMemsetAsync(c->d_delta, 0, (size_t)dn * sizeof(psk::DeltaSlot), c->stream) ==
                 cudaSuccess &&
             cudaMemsetAsync(c->d_err, 0, sizeof(uint32_t), c->stream) == cudaSuccess &&
             cudaMemsetAsync(c->d_stats, 0, kNumStats * sizeof(unsigned long long), c->stream) == cudaSuccess;
  for (psk::StateSoA* s : {&c->st, &c->pend}) {
    set = set && cudaMemsetAsync(s->b, 0, I * 4, c->stream) == cudaSuccess &&
          cudaMemsetAsync(s->qr, 0, I * 4, c->stream) == cudaSuccess &&
          cudaMemsetAsync(s->q, 0, I * 8, c->stream) == cudaSuccess &&
          cudaMemsetAsync(s->S, 0, I * 8, c->stream) == cudaSuccess &&
          cudaMemsetAsync(s->M, 0, I * 8, c->stream) == cudaSuccess &&
          cudaMemsetAsync(s->Bmax, 0, I * 4, c->stream) == cudaSuccess;
  }
  set = set && cudaMemcpyAsync(c->d_cap, c->cap.data(), I * sizeof(uint64_t), cudaMemcpyHostToDevice, c->stream) ==
                   cudaSuccess;
  if (c->lru)
    set = set && cudaMemsetAsync(c->meta.last_use, 0, c->total_slots * 4, c->stream) == cudaSuccess &&
          cudaMemsetAsync(c->meta.children, 0, c->total_slots * 4, c->stream) == cudaSuccess &&
          cudaMemsetAsync(c->meta.parent, 0xFF, c->total_slots * 8, c->stream) == cudaSuccess;  // kNoParent
  if (c->rq.M)
    set = set && cudaMemsetAsync(c->rq.q_head, 0, I * 4, c->stream) == cudaSuccess &&
          cudaMemsetAsync(c->rq.q_len, 0, I * 4, c->stream) == cudaSuccess &&
          cudaMemsetAsync(c->rq.d_len, 0, I * 4, c->stream) == cudaSuccess;
  if (!set || cudaStreamSynchronize(c->stream) != cudaSuccess) return bail(PS_ERR_CUDA);
  c->probe_grid = pskl::probe_max_grid(c->I, c->num_sms);
  if (cudaGetLastError() != cudaSuccess) return bail(PS_ERR_CUDA);
  *out = c;
  return PS_OK;
}

void ps_destroy(ps_ctx* c) {
  if (!c) return;
  {
    DeviceGuard g(c->device);
    if (c->stream) cudaStreamSynchronize(c->stream);
    for (void* p : c->allocs) cudaFree(p);
    if (c->h_err) cudaFreeHost(c->h_err);
    if (c->h_more) cudaFreeHost(c->h_more);
    for (cudaEvent_t e : c->ev)
      if (e) cudaEventDestroy(e);
    if (c->own_stream && c->stream) cudaStreamDestroy(c->stream);
  }
  delete c;
}

const char* ps_last_error(const ps_ctx* c) { return c ? c->err.c_str() : "null context"; }

ps_status ps_load_instances(ps_ctx* c, const ps_instance_state* s, uint32_t n) {
  if (!c) return PS_ERR_INVALID;
  c->shard_pending = false;
  if (!s || n != c->I) return fail(c, PS_ERR_INVALID, "need exactly num_instances states");
  const uint32_t I = c->I;
  std::vector<int32_t> b(I), qr(I), bm(I);
  std::vector<int64_t> q(I), S(I), M(I);
  for (uint32_t i = 0; i < I; ++i) {
    const ps_instance_state& x = s[i];
    if (x.b < 0 || x.b >= (1 << 17) || x.qr < 0 || x.qr >= (1 << 17) || x.q_tokens < 0 ||
        x.q_tokens >= (1ll << 40) || x.S_tokens < 0 || x.S_tokens >= (1ll << 50) || x.M_KV_tokens < 0 ||
        x.M_KV_tokens >= (1ll << 50) || x.B_max < 0)
      return fail(c, PS_ERR_INVALID, "instance " + std::to_string(i) + ": state out of range");
    b[i] = x.b; qr[i] = x.qr; q[i] = x.q_tokens; S[i] = x.S_tokens; M[i] = x.M_KV_tokens; bm[i] = x.B_max;
  }
  DeviceGuard g(c->device);
  c->pending = false;
  PS_TRY_CUDA(c, cudaMemcpyAsync(c->st.b, b.data(), I * 4, cudaMemcpyHostToDevice, c->stream));
  PS_TRY_CUDA(c, cudaMemcpyAsync(c->st.qr, qr.data(), I * 4, cudaMemcpyHostToDevice, c->stream));
  PS_TRY_CUDA(c, cudaMemcpyAsync(c->st.q, q.data(), I * 8, cudaMemcpyHostToDevice, c->stream));
  PS_TRY_CUDA(c, cudaMemcpyAsync(c->st.S, S.data(), I * 8, cudaMemcpyHostToDevice, c->stream));
  PS_TRY_CUDA(c, cudaMemcpyAsync(c->st.M, M.data(), I * 8, cudaMemcpyHostToDevice, c->stream));
  PS_TRY_CUDA(c, cudaMemcpyAsync(c->st.Bmax, bm.data(), I * 4, cudaMemcpyHostToDevice, c->stream));
  PS_TRY_CUDA(c, cudaStreamSynchronize(c->stream));
  return PS_OK;
}

static ps_status read_state(ps_ctx* c, const psk::StateSoA& st, ps_instance_state* out, uint32_t n) {
  if (!out || n != c->I) return fail(c, PS_ERR_INVALID, "need exactly num_instances states");
  const uint32_t I = c->I;
  std::vector<int32_t> b(I), qr(I), bm(I);
  std::vector<int64_t> q(I), S(I), M(I);
  DeviceGuard g(c->device);
  PS_TRY_CUDA(c, cudaMemcpyAsync(b.data(), st.b, I * 4, cudaMemcpyDeviceToHost, c->stream));
  PS_TRY_CUDA(c, cudaMemcpyAsync(qr.data(), st.qr, I * 4, cudaMemcpyDeviceToHost, c->stream));
  PS_TRY_CUDA(c, cudaMemcpyAsync(q.data(), st.q, I * 8, cudaMemcpyDeviceToHost, c->stream));
  PS_TRY_CUDA(c, cudaMemcpyAsync(S.data(), st.S, I * 8, cudaMemcpyDeviceToHost, c->stream));
  PS_TRY_CUDA(c, cudaMemcpyAsync(M.data(), st.M, I * 8, cudaMemcpyDeviceToHost, c->stream));
  PS_TRY_CUDA(c, cudaMemcpyAsync(bm.data(), st.Bmax, I * 4, cudaMemcpyDeviceToHost, c->stream));
  PS_TRY_CUDA(c, cudaStreamSynchronize(c->stream));
  for (uint32_t i = 0; i < I; ++i) {
    out[i].b = b[i]; out[i].qr = qr[i]; out[i].q_tokens = q[i]; out[i].S_tokens = S[i];
    out[i].M_KV_tokens = M[i]; out[i].B_max = bm[i];
  }
  return PS_OK;
}

ps_status ps_get_instances(ps_ctx* c, ps_instance_state* out, uint32_t n) {
  if (!c) return PS_ERR_INVALID;
  return read_state(c, c->st, out, n);
}

ps_status ps_calibrate(ps_ctx* c, uint32_t n, const int32_t* batch, const int64_t* ctx_tokens,
                       const float* measured_ms, float weight) {
  if (!c) return PS_ERR_INVALID;
  c->shard_pending = false;
  if (!(weight > 0.0f && weight <= 1.0f)) return fail(c, PS_ERR_INVALID, "calibration weight must be in (0, 1]");
  if (n == 0) return PS_OK;
  if (!batch || !ctx_tokens || !measured_ms) return fail(c, PS_ERR_INVALID, "NULL calibration sample array");
  for (uint32_t k = 0; k < n; ++k)
    if (batch[k] < 0 || ctx_tokens[k] < 0 || !std::isfinite(measured_ms[k]) || !(measured_ms[k] > 0.0f))
      return fail(c, PS_ERR_INVALID, "calibration sample " + std::to_string(k) +
                                         ": batch and context >= 0, duration finite and > 0");
  psk::DevModel& m = c->model;
  pscal::ema_update(m.b0, m.b1, m.b2, m.nseg, m.seg_lo, m.ema, n, batch, ctx_tokens, measured_ms, weight);
  return PS_OK;
}

ps_status ps_get_ema_factors(ps_ctx* c, float* out, uint32_t n) {
  if (!c) return PS_ERR_INVALID;
  if (!out || n < (uint32_t)c->model.nseg) return fail(c, PS_ERR_INVALID, "need nseg entries");
  for (int s = 0; s < c->model.nseg; ++s) out[s] = c->model.ema[s];
  return PS_OK;
}

ps_status ps_set_model(ps_ctx* c, const ps_model* m) {
  if (!c) return PS_ERR_INVALID;
  c->shard_pending = false;
  if (!m) return fail(c, PS_ERR_INVALID, "NULL model");
  if (check_model(c, *m) != PS_OK) return PS_ERR_INVALID;
  c->model = to_dev(*m);
  return PS_OK;
}

ps_status ps_set_wait_limit(ps_ctx* c, uint64_t ns) {
  if (!c) return PS_ERR_INVALID;
  if (ns > 60ull * kDefaultWaitNs) return fail(c, PS_ERR_INVALID, "wait limit above 60 s");
  c->gsync.wait_ns = ns == 0 ? kDefaultWaitNs : ns;
  return PS_OK;
}

ps_status ps_get_pending_instances(ps_ctx* c, ps_instance_state* out, uint32_t n) {
  if (!c) return PS_ERR_INVALID;
  if (!c->pending) return fail(c, PS_ERR_STATE, "no pending window");
  return read_state(c, c->pend, out, n);
}

ps_status ps_insert_chains(ps_ctx* c, uint64_t nchains, const uint32_t* inst, const uint64_t* off,
                           const uint64_t* hash, const uint64_t* parent, uint32_t last_use, int32_t on_device) {
  if (!c) return PS_ERR_INVALID;
  c->shard_pending = false;
  if (nchains == 0) return PS_OK;
  if (!inst || !off || !parent || (on_device != 0 && on_device != 1))
    return fail(c, PS_ERR_INVALID, "bad chain arrays");
  DeviceGuard g(c->device);
  uint64_t total = 0;
  const uint32_t* d_inst = inst;
  const uint64_t* d_off = off;
  const uint64_t* d_hash = hash;
  const uint64_t* d_parent = parent;
  void* tmp = nullptr;
  if (!on_device) {
    if (off[0] != 0) return fail(c, PS_ERR_INVALID, "off[0] must be 0");
    for (uint64_t k = 0; k < nchains; ++k) {
      if (off[k + 1] < off[k]) return fail(c, PS_ERR_INVALID, "off must ascend");
      if (inst[k] >= c->I) return fail(c, PS_ERR_INVALID, "instance id out of range");
    }
    total = off[nchains];
    if (total && !hash) return fail(c, PS_ERR_INVALID, "hash is NULL");
    const size_t bytes = nchains * 4 + (nchains + 1) * 8 + nchains * 8 + total * 8 + 16;
    PS_TRY_CUDA(c, cudaMalloc(&tmp, bytes));
    uint64_t* t_off = static_cast<uint64_t*>(tmp);
    uint64_t* t_parent = t_off + nchains + 1;
    uint64_t* t_hash = t_parent + nchains;
    uint32_t* t_inst = reinterpret_cast<uint32_t*>(t_hash + total);
    cudaError_t e = cudaMemcpyAsync(t_off, off, (nchains + 1) * 8, cudaMemcpyHostToDevice, c->stream);
    if (e == cudaSuccess) e = cudaMemcpyAsync(t_parent, parent, nchains * 8, cudaMemcpyHostToDevice, c->stream);
    if (e == cudaSuccess && total) e = cudaMemcpyAsync(t_hash, hash, total * 8, cudaMemcpyHostToDevice, c->stream);
    if (e == cudaSuccess) e = cudaMemcpyAsync(t_inst, inst, nchains * 4, cudaMemcpyHostToDevice, c->stream);
    if (e != cudaSuccess) {
      cudaFree(tmp);
      return fail(c, PS_ERR_CUDA, std::string("copy chains: ") + cudaGetErrorString(e));
    }
    d_off = t_off;
    d_hash = t_hash;
    d_inst = t_inst;
    d_parent = t_parent;
  } else {
    PS_TRY_CUDA(c, cudaMemcpy(&total, off + nchains, 8, cudaMemcpyDeviceToHost));
  }
  cudaError_t e = pskl::launch_insert_chains(c->d_slots, c->d_ovf, c->d_tdesc, c->I, c->d_count, nchains, d_inst, d_off,
                                             d_hash, d_parent, total, c->meta, last_use, c->d_err, c->num_sms,
                                             c->stream);
  if (e == cudaSuccess && c->search)
    e = pskl::launch_check_parents(c->d_slots, c->d_ovf, c->d_tdesc, c->I, nchains, d_inst, d_parent, c->d_err, c->num_sms,
                                   c->stream);
  ps_status s = e == cudaSuccess ? finish(c) : fail(c, PS_ERR_CUDA, cudaGetErrorString(e));
  if (tmp) cudaFree(tmp);
  if (s != PS_OK) return s;
  return check_capacity(c);
}

ps_status ps_insert_blocks(ps_ctx* c, uint32_t inst, const uint64_t* chain, uint64_t n, uint64_t parent_hash,
                           uint32_t last_use) {
  if (!c) return PS_ERR_INVALID;
  c->shard_pending = false;
  if (n == 0) return PS_OK;
  const uint64_t off[2] = {0, n};
  return ps_insert_chains(c, 1, &inst, off, chain, &parent_hash, last_use, 0);
}

ps_status ps_cached_blocks(ps_ctx* c, uint64_t* out, uint32_t n) {
  if (!c) return PS_ERR_INVALID;
  if (!out || n != c->I) return fail(c, PS_ERR_INVALID, "need num_instances entries");
  DeviceGuard g(c->device);
  PS_TRY_CUDA(c, cudaMemcpyAsync(out, c->d_count, n * 8, cudaMemcpyDeviceToHost, c->stream));
  PS_TRY_CUDA(c, cudaStreamSynchronize(c->stream));
  return PS_OK;
}

ps_status ps_score_window(ps_ctx* c, const ps_window* w, ps_scores* out) {
  if (!c) return PS_ERR_INVALID;
  if (out && out->outputs_on_device != 0 && out->outputs_on_device != 1)
    return fail(c, PS_ERR_INVALID, "outputs_on_device must be 0 or 1");
  DeviceGuard g(c->device);
  reset_timers(c);
  psk::WindowDev wd{};
  ps_status s = stage_window(c, w, &wd);
  if (s != PS_OK) return s;
  uint32_t* hits = nullptr;
  s = run_probe_and_score(c, wd, out, &hits);
  if (s != PS_OK) return s;
  return finish(c);
}

ps_status ps_shard_wmin(ps_ctx* c, const ps_window* w, uint32_t* wmin_ord, int32_t on_device) {
  if (!c) return PS_ERR_INVALID;
  if (on_device != 0 && on_device != 1) return fail(c, PS_ERR_INVALID, "on_device must be 0 or 1");
  DeviceGuard g(c->device);
  reset_timers(c);
  psk::WindowDev wd{};
  ps_status s = stage_window(c, w, &wd);
  if (s != PS_OK) return s;
  if (wd.R > 0 && !wmin_ord) return fail(c, PS_ERR_INVALID, "wmin_ord is NULL");
  uint32_t* hits = nullptr;
  s = run_probe_and_score(c, wd, nullptr, &hits);  // the probe phase only: hits into the context's buffer
  if (s != PS_OK) return s;
  psk::ShardIO sh;
  sh.wmin_out = on_device ? wmin_ord : c->d_shard_wmin;
  record(c, kEvScore0);
  PS_TRY_CUDA(c, pskl::launch_score(hits, c->st, c->I, wd, c->model, nullptr, nullptr, nullptr, nullptr, nullptr,
                                    c->num_sms, c->stream, sh));
  record(c, kEvScore1);
  c->ev_used[1] = true;
  if (!on_device) PS_TRY_CUDA(c, deliver(c, wmin_ord, c->d_shard_wmin, wd.R, 0));
  s = finish(c);
  if (s != PS_OK) return s;
  c->shard_pending = true;
  c->shard_win = wd;
  return PS_OK;
}

ps_status ps_shard_pick(ps_ctx* c, const uint32_t* wmin_ord, uint32_t id_base, uint64_t* key, uint32_t* tie,
                        int32_t on_device, ps_scores* opt) {
  if (!c) return PS_ERR_INVALID;
  if (!c->shard_pending) return fail(c, PS_ERR_STATE, "no window from ps_shard_wmin (or the context changed since)");
  if (on_device != 0 && on_device != 1) return fail(c, PS_ERR_INVALID, "on_device must be 0 or 1");
  if (opt && opt->outputs_on_device != 0 && opt->outputs_on_device != 1)
    return fail(c, PS_ERR_INVALID, "outputs_on_device must be 0 or 1");
  const psk::WindowDev wd = c->shard_win;
  if (wd.R > 0 && (!wmin_ord || !key || !tie)) return fail(c, PS_ERR_INVALID, "wmin_ord, key and tie are required");
  if ((uint64_t)id_base + c->I > (c->model.sel == psk::kSelHCQ ? 4096ull : 0x7FFFFFFFull))
    return fail(c, PS_ERR_INVALID, "id_base + num_instances too large (4096 under H-C-Q)");
  DeviceGuard g(c->device);
  for (bool& u : c->ev_used) u = false;
  c->probe_split = false;
  psk::ShardIO sh;
  sh.id_base = id_base;
  if (on_device) {
    sh.wmin_in = wmin_ord;
    sh.key_out = reinterpret_cast<unsigned long long*>(key);
    sh.tie_out = tie;
  } else {
    if (wd.R) PS_TRY_CUDA(c, cudaMemcpyAsync(c->d_shard_wmin, wmin_ord, wd.R * sizeof(uint32_t), cudaMemcpyHostToDevice,
                                             c->stream));
    sh.wmin_in = c->d_shard_wmin;
    sh.key_out = c->d_shard_key;
    sh.tie_out = c->d_shard_tie;
  }
  const int dev_out = opt ? opt->outputs_on_device : 0;
  const size_t RI = (size_t)wd.R * c->I;
  float* tpot = (opt && opt->tpot) ? (dev_out ? opt->tpot : c->d_tpot_o) : nullptr;
  float* ttft = (opt && opt->ttft) ? (dev_out ? opt->ttft : c->d_ttft_o) : nullptr;
  uint8_t* cls = (opt && opt->cls) ? (dev_out ? opt->cls : c->d_cls) : nullptr;
  int32_t* best = (opt && opt->best) ? (dev_out ? opt->best : c->d_best) : nullptr;
  uint8_t* path = (opt && opt->path) ? (dev_out ? opt->path : c->d_path) : nullptr;
  record(c, kEvScore0);
  PS_TRY_CUDA(c, pskl::launch_score(c->d_hits, c->st, c->I, wd, c->model, tpot, ttft, cls, best, path, c->num_sms,
                                    c->stream, sh));
  record(c, kEvScore1);
  c->ev_used[1] = true;
  if (!on_device) {
    PS_TRY_CUDA(c, deliver(c, reinterpret_cast<unsigned long long*>(key), c->d_shard_key, wd.R, 0));
    PS_TRY_CUDA(c, deliver(c, tie, c->d_shard_tie, wd.R, 0));
  }
  if (opt) {
    PS_TRY_CUDA(c, deliver(c, opt->hits, c->d_hits, RI, dev_out));
    if (!dev_out) {
      PS_TRY_CUDA(c, deliver(c, opt->tpot, c->d_tpot_o, RI, 0));
      PS_TRY_CUDA(c, deliver(c, opt->ttft, c->d_ttft_o, RI, 0));
      PS_TRY_CUDA(c, deliver(c, opt->cls, c->d_cls, RI, 0));
      PS_TRY_CUDA(c, deliver(c, opt->best, c->d_best, wd.R, 0));
      PS_TRY_CUDA(c, deliver(c, opt->path, c->d_path, wd.R, 0));
    }
  }
  return finish(c);
}

ps_status ps_schedule_window(ps_ctx* c, const ps_window* w, ps_decisions* out, ps_scores* opt_scores) {
  if (!c) return PS_ERR_INVALID;
  if (out && out->outputs_on_device != 0 && out->outputs_on_device != 1)
    return fail(c, PS_ERR_INVALID, "outputs_on_device must be 0 or 1");
  if (opt_scores && opt_scores->outputs_on_device != 0 && opt_scores->outputs_on_device != 1)
    return fail(c, PS_ERR_INVALID, "outputs_on_device must be 0 or 1");
  DeviceGuard g(c->device);
  reset_timers(c);
  c->pending = false;
  psk::WindowDev wd{};
  ps_status s = stage_window(c, w, &wd);
  if (s != PS_OK) return s;
  uint32_t* hit0 = nullptr;
  s = run_probe_and_score(c, wd, opt_scores, &hit0);
  if (s != PS_OK) return s;
  record(c, kEvGreedy0);
  if (c->search) {
    PS_TRY_CUDA(c, pskl::launch_greedy_search(c->d_rows, wd, c->I, hit0, c->d_tpf, c->st, c->pend, c->model, c->d_delta,
                                              c->delta_nslots, c->d_assign, c->d_dpath, c->d_hchosen, c->d_err,
                                              c->gsync, c->stream));
  } else {
    PS_TRY_CUDA(c, pskl::launch_greedy(c->d_slots, c->d_ovf, c->d_tdesc, c->I, wd, hit0, c->st, c->pend, c->model,
                                       c->d_delta, c->delta_nslots, c->d_assign, c->d_dpath, c->d_hchosen, c->d_err,
                                       0, c->stream));
  }
  record(c, kEvGreedy1);
  c->ev_used[2] = true;
  PS_TRY_CUDA(c, pskl::launch_delta_clear(c->d_delta, c->delta_nslots, c->stream));
  if (out) {
    PS_TRY_CUDA(c, deliver(c, out->assign, c->d_assign, wd.R, out->outputs_on_device));
    PS_TRY_CUDA(c, deliver(c, out->path, c->d_dpath, wd.R, out->outputs_on_device));
    PS_TRY_CUDA(c, deliver(c, out->hit_chosen, c->d_hchosen, wd.R, out->outputs_on_device));
  }
  s = finish(c);
  if (s != PS_OK) return s;
  c->pending = true;
  c->pend_win = wd;
  return PS_OK;
}

ps_status ps_commit_window(ps_ctx* c, uint32_t last_use) {
  if (!c) return PS_ERR_INVALID;
  c->shard_pending = false;
  if (!c->pending) return fail(c, PS_ERR_STATE, "no pending window");
  if (c->rq.M && c->pend_win.R && !c->pend_out)
    return fail(c, PS_ERR_INVALID, "request tracking needs the window's out_tokens");
  DeviceGuard g(c->device);
  record(c, kEvCommit0);
  PS_TRY_CUDA(c, pskl::launch_commit(c->d_slots, c->d_ovf, c->d_tdesc, c->I, c->d_count, c->pend_win, c->d_assign,
                                     c->d_hchosen, c->meta, last_use, c->rq, c->pend_out, c->d_cprefix, c->d_err,
                                     c->num_sms, c->stream));
  const size_t I = c->I;
  PS_TRY_CUDA(c, cudaMemcpyAsync(c->st.b, c->pend.b, I * 4, cudaMemcpyDeviceToDevice, c->stream));
  PS_TRY_CUDA(c, cudaMemcpyAsync(c->st.qr, c->pend.qr, I * 4, cudaMemcpyDeviceToDevice, c->stream));
  PS_TRY_CUDA(c, cudaMemcpyAsync(c->st.q, c->pend.q, I * 8, cudaMemcpyDeviceToDevice, c->stream));
  PS_TRY_CUDA(c, cudaMemcpyAsync(c->st.S, c->pend.S, I * 8, cudaMemcpyDeviceToDevice, c->stream));
  PS_TRY_CUDA(c, cudaMemcpyAsync(c->st.M, c->pend.M, I * 8, cudaMemcpyDeviceToDevice, c->stream));
  PS_TRY_CUDA(c, cudaMemcpyAsync(c->st.Bmax, c->pend.Bmax, I * 4, cudaMemcpyDeviceToDevice, c->stream));
  record(c, kEvCommit1);
  c->ev_used[3] = true;
  c->pending = false;
  return finish(c);
}

ps_status ps_load_requests(ps_ctx* c, uint64_t n, const uint32_t* inst, const uint32_t* state, const uint32_t* L,
                           const uint32_t* out, const uint64_t* rem) {
  if (!c) return PS_ERR_INVALID;
  c->shard_pending = false;
  if (!c->rq.M) return fail(c, PS_ERR_STATE, "context has no request tracking (max_active_requests = 0)");
  if (n && (!inst || !state || !L || !out || !rem)) return fail(c, PS_ERR_INVALID, "request array is NULL");
  const uint32_t I = c->I, M = c->rq.M;
  const size_t IM = (size_t)I * M;
  std::vector<uint32_t> qlen(I, 0), dlen(I, 0), qL(IM), qo(IM), dL(IM), dO(IM), dR(IM);
  std::vector<uint64_t> qR(IM);
  std::vector<int32_t> b(I, 0), qr(I, 0);
  std::vector<int64_t> q(I, 0), S(I, 0);
  for (uint64_t k = 0; k < n; ++k) {
    const uint32_t i = inst[k];
    if (i >= I || state[k] > 1) return fail(c, PS_ERR_INVALID, "request " + std::to_string(k) + ": bad instance or state");
    if (state[k] == 0) {
      if (qlen[i] >= M) return fail(c, PS_ERR_CAPACITY, "too many queued requests on instance " + std::to_string(i));
      const size_t at = (size_t)i * M + qlen[i]++;
      qL[at] = L[k]; qo[at] = out[k]; qR[at] = rem[k];
      qr[i] += 1; q[i] += (int64_t)rem[k]; S[i] += L[k];
    } else {
      if (rem[k] < 1 || rem[k] > out[k]) return fail(c, PS_ERR_INVALID, "decoding request needs 1 <= rem <= out");
      if (dlen[i] >= M) return fail(c, PS_ERR_CAPACITY, "too many decoding requests on instance " + std::to_string(i));
      const size_t at = (size_t)i * M + dlen[i]++;
      dL[at] = L[k]; dO[at] = out[k]; dR[at] = (uint32_t)rem[k];
      b[i] += 1; S[i] += (int64_t)L[k] + (int64_t)(out[k] - (uint32_t)rem[k]);
    }
  }
  DeviceGuard g(c->device);
  c->pending = false;
  std::vector<uint32_t> zero(I, 0);
  PS_TRY_CUDA(c, cudaMemcpyAsync(c->rq.q_head, zero.data(), I * 4, cudaMemcpyHostToDevice, c->stream));
  PS_TRY_CUDA(c, cudaMemcpyAsync(c->rq.q_len, qlen.data(), I * 4, cudaMemcpyHostToDevice, c->stream));
  PS_TRY_CUDA(c, cudaMemcpyAsync(c->rq.d_len, dlen.data(), I * 4, cudaMemcpyHostToDevice, c->stream));
  PS_TRY_CUDA(c, cudaMemcpyAsync(c->rq.q_L, qL.data(), IM * 4, cudaMemcpyHostToDevice, c->stream));
  PS_TRY_CUDA(c, cudaMemcpyAsync(c->rq.q_out, qo.data(), IM * 4, cudaMemcpyHostToDevice, c->stream));
  PS_TRY_CUDA(c, cudaMemcpyAsync(c->rq.q_rem, qR.data(), IM * 8, cudaMemcpyHostToDevice, c->stream));
  PS_TRY_CUDA(c, cudaMemcpyAsync(c->rq.d_L, dL.data(), IM * 4, cudaMemcpyHostToDevice, c->stream));
  PS_TRY_CUDA(c, cudaMemcpyAsync(c->rq.d_out, dO.data(), IM * 4, cudaMemcpyHostToDevice, c->stream));
  PS_TRY_CUDA(c, cudaMemcpyAsync(c->rq.d_rem, dR.data(), IM * 4, cudaMemcpyHostToDevice, c->stream));
  PS_TRY_CUDA(c, cudaMemcpyAsync(c->st.b, b.data(), I * 4, cudaMemcpyHostToDevice, c->stream));
  PS_TRY_CUDA(c, cudaMemcpyAsync(c->st.qr, qr.data(), I * 4, cudaMemcpyHostToDevice, c->stream));
  PS_TRY_CUDA(c, cudaMemcpyAsync(c->st.q, q.data(), I * 8, cudaMemcpyHostToDevice, c->stream));
  PS_TRY_CUDA(c, cudaMemcpyAsync(c->st.S, S.data(), I * 8, cudaMemcpyHostToDevice, c->stream));
  PS_TRY_CUDA(c, cudaStreamSynchronize(c->stream));
  return PS_OK;
}

ps_status ps_advance_window(ps_ctx* c, const ps_advance_params* p) {
  if (!c) return PS_ERR_INVALID;
  c->shard_pending = false;
  if (!p || !(p->window_ms > 0.0f) || !std::isfinite(p->window_ms) || (p->evict != 0 && p->evict != 1))
    return fail(c, PS_ERR_INVALID, "advance params: window_ms > 0, evict 0 or 1");
  if (c->pending) return fail(c, PS_ERR_STATE, "commit the pending window before advancing");
  if (!c->rq.M) return fail(c, PS_ERR_STATE, "context has no request tracking (max_active_requests = 0)");
  if (p->evict && !c->lru) return fail(c, PS_ERR_STATE, "eviction needs track_lru");
  DeviceGuard g(c->device);
  PS_TRY_CUDA(c, pskl::launch_advance(c->st, c->I, c->rq, c->model, p->window_ms, p->prefill_tokens, c->d_err,
                                      c->stream));
  if (p->evict)
    PS_TRY_CUDA(c, pskl::launch_evict(c->d_slots, c->d_tdesc, c->I, c->d_count, c->d_cap, c->meta, c->d_leafbuf,
                                      c->d_nleaf, c->d_more, c->h_more, c->max_instance_slots, c->d_err, c->stream));
  return finish(c);
}

ps_status ps_last_timings(ps_ctx* c, float* ms, uint32_t n) {
  if (!c) return PS_ERR_INVALID;
  if (!ms || n < 4) return fail(c, PS_ERR_INVALID, "need 4 entries");
  DeviceGuard g(c->device);
  auto span = [&](int a, int b) {
    float t = 0.0f;
    return cudaEventElapsedTime(&t, c->ev[a], c->ev[b]) == cudaSuccess ? t : -1.0f;
  };
  for (int k = 0; k < kNumPhases; ++k) ms[k] = c->ev_used[k] ? span(2 * k, 2 * k + 1) : -1.0f;
  const int split[3][2] = {{kEvProbe0, kEvRelDone}, {kEvRelDone, kEvProbeMid}, {kEvProbeMid, kEvProbe1}};
  for (uint32_t k = 0; k < 3 && 4 + k < n; ++k)
    ms[4 + k] = (c->ev_used[0] && c->probe_split) ? span(split[k][0], split[k][1]) : -1.0f;
  return PS_OK;
}

ps_status ps_last_probe_stats(ps_ctx* c, uint64_t* out, uint32_t n) {
  if (!c) return PS_ERR_INVALID;
  if (!out || n < (uint32_t)kNumStats) return fail(c, PS_ERR_INVALID, "need 6 entries");
  DeviceGuard g(c->device);
  unsigned long long v[kNumStats] = {};
  unsigned long long gs[psk::kGreedyStats] = {};
  if (c->ev_used[0]) PS_TRY_CUDA(c, cudaMemcpyAsync(v, c->d_stats, sizeof(v), cudaMemcpyDeviceToHost, c->stream));
  if (c->ev_used[2] && c->search && n >= 8)
    PS_TRY_CUDA(c, cudaMemcpyAsync(gs, c->gsync.stats, sizeof(gs), cudaMemcpyDeviceToHost, c->stream));
  PS_TRY_CUDA(c, cudaStreamSynchronize(c->stream));
  for (int k = 0; k < kNumStats; ++k) out[k] = v[k];
  for (uint32_t k = 0; k < (uint32_t)psk::kGreedyStats && 6 + k < n; ++k) out[6 + k] = gs[k];
  return PS_OK;
}

}  // extern "C"
