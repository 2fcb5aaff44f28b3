// Allocation-free scoring entry point (ps_score_window_noalloc).
//
// For callers that may not allocate device memory at all: a serving process whose memory manager
// reserves the device up front (so the KV cache can take the rest) and forbids allocations
// afterwards, or a scheduler loop that must never call cudaMalloc because an allocation can
// synchronise the device and stall the serving streams.  Such a caller owns every buffer: it passes
// the cache tables, the instance state, the window and the outputs, all in device memory.
//
// The probe kernel's hit matrix is the only intermediate buffer; here it lives in the file-scope
// array below, which every GPU that loads the library holds until the process exits.  Host code
// cannot use the array's name as a device address: on each device the first call looks the address
// up with cudaGetSymbolAddress (with that device current) and passes the pointer to the kernels.
#include <mutex>

#include "packserve.h"
#include "ps_internal.cuh"

namespace {

constexpr uint64_t kMaxPairs = PS_NOALLOC_MAX_PAIRS;
constexpr uint64_t kErrWordIndex = kMaxPairs;  // one u32 after the hit matrix
constexpr int kMaxDevices = 64;

static __device__ __align__(256) uint32_t g_noalloc_scratch[kMaxPairs + 64];

struct DeviceScratch {
  bool ready = false;
  uint32_t* base = nullptr;  // device address of g_noalloc_scratch on this device
  int num_sms = 0;
  int probe_grid_small = 0;  // probe grid for I < 64 (4-warp blocks)
  int probe_grid_large = 0;  // probe grid for I >= 64 (8-warp blocks)
};

std::mutex g_mu;
DeviceScratch g_dev[kMaxDevices];

// One-time set-up for the current device: resolve the array's device address and the launch shapes.
ps_status setup(int dev, DeviceScratch** out) {
  if (dev < 0 || dev >= kMaxDevices) return PS_ERR_INVALID;
  std::lock_guard<std::mutex> lock(g_mu);
  DeviceScratch& d = g_dev[dev];
  if (!d.ready) {
    void* p = nullptr;
    if (cudaGetSymbolAddress(&p, g_noalloc_scratch) != cudaSuccess || p == nullptr) return PS_ERR_CUDA;
    if (cudaDeviceGetAttribute(&d.num_sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess) return PS_ERR_CUDA;
    d.probe_grid_small = pskl::probe_max_grid(1, d.num_sms);
    d.probe_grid_large = pskl::probe_max_grid(64, d.num_sms);
    if (cudaGetLastError() != cudaSuccess) return PS_ERR_CUDA;
    d.base = static_cast<uint32_t*>(p);
    d.ready = true;
  }
  *out = &d;
  return PS_OK;
}

bool model_ok(const ps_model& m) {
  const float c[] = {m.a0, m.a1, m.a2, m.a3, m.a4, m.a5, m.b0, m.b1, m.b2, m.g_q, m.eta, m.lout_median};
  for (float x : c)
    if (!(x == x) || x > 1e9f || x < -1e9f) return false;
  if (m.eta < 0.0f || (m.interference_mode != 0 && m.interference_mode != 1) ||
      (m.ttft_filter != 0 && m.ttft_filter != 1) || m.nseg < 1 || m.nseg > PS_MAX_EMA_SEGMENTS || m.seg_lo[0] > 1)
    return false;
  for (int s = 0; s < m.nseg; ++s) {
    if (!(m.ema_factor[s] > 0.0f && m.ema_factor[s] <= 1e9f)) return false;
    if (s > 0 && m.seg_lo[s] <= m.seg_lo[s - 1]) return false;
  }
  if ((m.cache_filter_off | m.slo_filter_off | m.fallback_dcq) & ~1) return false;
  return m.selector >= PS_SELECT_DCQ && m.selector <= PS_SELECT_HCQ;
}

psk::DevModel dev_model(const ps_model& m) {
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

static_assert(sizeof(ps_table_desc) == sizeof(psk::TableDesc), "ps_table_desc layout");

// The caller's table descriptors live in device memory: before any lookup reads a table, check that
// each starts on a whole bucket (the probe reads a bucket as four 16-byte loads) and has at least
// one bucket.  A bad descriptor sets the error word, so the call returns PS_ERR_INVALID instead of
// reading misaligned or absent slots.
__global__ void check_tables_kernel(const psk::TableDesc* __restrict__ td, uint32_t I, uint32_t* err) {
  for (uint32_t i = blockIdx.x * blockDim.x + threadIdx.x; i < I; i += gridDim.x * blockDim.x) {
    const psk::TableDesc d = td[i];
    if (d.nbkt == 0u || (d.base % psk::kBucketSlots) != 0u) atomicOr(err, psk::kErrTableLayout);
  }
}

}  // namespace

extern "C" {

ps_status ps_score_window_noalloc(const uint64_t* slots, const uint64_t* overflow_bits, const ps_table_desc* tables,
                                  uint32_t num_instances,
                                  const ps_state_arrays* state, const ps_window* w, const ps_model* model,
                                  int32_t probe_mode, ps_scores* out, void* cuda_stream) {
  if (!slots || !overflow_bits || !tables || !state || !w || !model || !out) return PS_ERR_INVALID;
  // buckets are read with 16-byte loads; overflow words and descriptors are 8-byte words
  if ((reinterpret_cast<uintptr_t>(slots) & 15u) || (reinterpret_cast<uintptr_t>(overflow_bits) & 7u) ||
      (reinterpret_cast<uintptr_t>(tables) & 7u))
    return PS_ERR_INVALID;
  if (num_instances < 1 || num_instances > 4096) return PS_ERR_INVALID;
  if (w->inputs_on_device != 1 || out->outputs_on_device != 1 || w->parent) return PS_ERR_INVALID;
  if (probe_mode != PS_PROBE_LINEAR && probe_mode != PS_PROBE_SEARCH) return PS_ERR_INVALID;
  if (!state->b || !state->qr || !state->q_tokens || !state->S_tokens || !state->M_KV_tokens || !state->B_max)
    return PS_ERR_INVALID;
  if (!w->chain_off || (w->R > 0 && (!w->prompt_tokens || !w->ttft_target || !w->tpot_target)))
    return PS_ERR_INVALID;
  if ((uint64_t)w->R * num_instances > kMaxPairs) return PS_ERR_INVALID;
  if (!model_ok(*model)) return PS_ERR_INVALID;
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return PS_ERR_CUDA;
  DeviceScratch* d = nullptr;
  ps_status st = setup(dev, &d);
  if (st != PS_OK) return st;
  if (w->R == 0) return PS_OK;
  cudaStream_t s = static_cast<cudaStream_t>(cuda_stream);
  uint32_t* hits = d->base;
  uint32_t* err = d->base + kErrWordIndex;
  // The error word keeps the previous call's value: clear it first.
  if (cudaMemsetAsync(err, 0, sizeof(uint32_t), s) != cudaSuccess) return PS_ERR_CUDA;
  const psk::WindowDev wd{w->chain_off, w->chain_hash, w->prompt_tokens, w->ttft_target, w->tpot_target, w->R};
  if (pskl::launch_validate_window(wd, ~0ull, err, s) != cudaSuccess) return PS_ERR_CUDA;
  const psk::TableDesc* td = reinterpret_cast<const psk::TableDesc*>(tables);
  check_tables_kernel<<<(num_instances + 255) / 256, 256, 0, s>>>(td, num_instances, err);
  if (cudaGetLastError() != cudaSuccess) return PS_ERR_CUDA;
  uint32_t herr = 0;
  uint64_t nblk = 0;
  if (cudaMemcpyAsync(&herr, err, sizeof(uint32_t), cudaMemcpyDeviceToHost, s) != cudaSuccess ||
      cudaMemcpyAsync(&nblk, w->chain_off + w->R, sizeof(uint64_t), cudaMemcpyDeviceToHost, s) != cudaSuccess ||
      cudaStreamSynchronize(s) != cudaSuccess)
    return PS_ERR_CUDA;
  if (herr != 0 || (nblk > 0 && !w->chain_hash)) return PS_ERR_INVALID;
  const int grid = num_instances >= 64 ? d->probe_grid_large : d->probe_grid_small;
  const psk::DevModel dm = dev_model(*model);
  if (pskl::launch_probe(slots, overflow_bits, td, num_instances, wd, nullptr, psk::RowList{nullptr, nullptr}, hits, nullptr, dm, grid,
                         probe_mode == PS_PROBE_SEARCH, nullptr, nullptr, s) != cudaSuccess)
    return PS_ERR_CUDA;
  const psk::StateSoA soa{const_cast<int32_t*>(state->b), const_cast<int32_t*>(state->qr),
                          const_cast<int64_t*>(state->q_tokens), const_cast<int64_t*>(state->S_tokens),
                          const_cast<int64_t*>(state->M_KV_tokens), const_cast<int32_t*>(state->B_max)};
  if (out->tpot || out->ttft || out->cls || out->best || out->path) {
    if (pskl::launch_score(hits, soa, num_instances, wd, dev_model(*model), out->tpot, out->ttft, out->cls,
                           out->best, out->path, d->num_sms, s) != cudaSuccess)
      return PS_ERR_CUDA;
  }
  if (out->hits &&
      cudaMemcpyAsync(out->hits, hits, (size_t)w->R * num_instances * sizeof(uint32_t), cudaMemcpyDeviceToDevice,
                      s) != cudaSuccess)
    return PS_ERR_CUDA;
  if (cudaStreamSynchronize(s) != cudaSuccess) return PS_ERR_CUDA;
  return PS_OK;
}

}  // extern "C"
