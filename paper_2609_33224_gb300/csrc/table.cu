// Table maintenance kernels: bulk insertion of cached chains, commit of a scheduled window, and the
// device-side window layout check.
#include "ps_internal.cuh"

namespace {

// Index c of the chain containing block position pos: off[c] <= pos < off[c+1].
__device__ __forceinline__ uint64_t chain_of(const uint64_t* __restrict__ off, uint64_t nchains, uint64_t pos) {
  uint64_t lo = 0, hi = nchains;  // invariant: off[lo] <= pos < off[hi]
  while (hi - lo > 1) {
    const uint64_t mid = (lo + hi) >> 1;
    if (__ldg(off + mid) <= pos) lo = mid; else hi = mid;
  }
  return lo;
}

// Warp-aggregated count of new insertions per instance.
__device__ __forceinline__ void count_inserted(unsigned long long* count, uint32_t inst, bool inserted,
                                               bool active) {
  const unsigned act = __ballot_sync(0xffffffffu, active);
  if (!active) return;
  const unsigned same = __match_any_sync(act, inst);
  const unsigned ins = __ballot_sync(act, inserted) & same;
  const int leader = __ffs(same) - 1;
  if ((int)(threadIdx.x & 31) == leader && ins) atomicAdd(count + inst, (unsigned long long)__popc(ins));
}

__global__ void insert_chains_kernel(uint64_t* slots, const psk::TableDesc* __restrict__ tdesc, uint32_t I,
                                     unsigned long long* count, uint64_t nchains,
                                     const uint32_t* __restrict__ inst, const uint64_t* __restrict__ off,
                                     const uint64_t* __restrict__ hash, uint64_t total, uint32_t* err) {
  const uint64_t stride = (uint64_t)gridDim.x * blockDim.x;
  // Every lane of a warp runs the same number of iterations, so the warp-level count is safe.
  const uint64_t start = blockIdx.x * (uint64_t)blockDim.x + threadIdx.x;
  const uint64_t warp_start = start - (threadIdx.x & 31);
  for (uint64_t base = warp_start; base < total; base += stride) {
    const uint64_t pos = base + (threadIdx.x & 31);
    bool active = pos < total;
    bool inserted = false;
    uint32_t i = 0;
    if (active) {
      const uint64_t c = chain_of(off, nchains, pos);
      i = __ldg(inst + c);
      const uint64_t key = __ldg(hash + pos);
      if (i >= I) {
        atomicOr(err, psk::kErrBadInstance);
        active = false;
      } else if (key == psk::kEmpty || key == psk::kTomb) {
        atomicOr(err, psk::kErrReservedHash);
        active = false;
      } else {
        const int res = psk::main_insert(slots, tdesc[i], key);
        if (res < 0) atomicOr(err, psk::kErrTableFull);
        inserted = res == 1;
      }
    }
    count_inserted(count, i, inserted, active);
  }
}

// Commit: each admitted request caches its uncached blocks chain[h..nb) on its instance.
__global__ void commit_kernel(uint64_t* slots, const psk::TableDesc* __restrict__ tdesc, uint32_t I,
                              unsigned long long* count, psk::WindowDev w, const int32_t* __restrict__ assign,
                              const uint32_t* __restrict__ hit_chosen, uint32_t* err) {
  const int lane = threadIdx.x & 31;
  const uint32_t warps_total = (gridDim.x * blockDim.x) >> 5;
  for (uint32_t r = (blockIdx.x * blockDim.x + threadIdx.x) >> 5; r < w.R; r += warps_total) {
    const int32_t j = assign[r];
    if (j < 0 || (uint32_t)j >= I) continue;
    const uint64_t o = w.off[r];
    const uint64_t nb = w.off[r + 1] - o;
    const psk::TableDesc d = tdesc[j];
    for (uint64_t base = hit_chosen[r]; base < nb; base += 32) {
      const uint64_t k = base + lane;
      bool inserted = false;
      if (k < nb) {
        const uint64_t key = w.hash[o + k];
        if (key != psk::kEmpty && key != psk::kTomb) {
          const int res = psk::main_insert(slots, d, key);
          if (res < 0) atomicOr(err, psk::kErrTableFull);
          inserted = res == 1;
        }
      }
      const unsigned ins = __ballot_sync(0xffffffffu, inserted);
      if (lane == 0 && ins) atomicAdd(count + j, (unsigned long long)__popc(ins));
    }
  }
}

// Prefix closure check (search mode): every chain's parent must be cached once the chains are in.
__global__ void check_parents_kernel(const uint64_t* slots, const psk::TableDesc* __restrict__ tdesc, uint32_t I,
                                     uint64_t nchains, const uint32_t* __restrict__ inst,
                                     const uint64_t* __restrict__ parent, uint32_t* err) {
  for (uint64_t c = blockIdx.x * (uint64_t)blockDim.x + threadIdx.x; c < nchains; c += (uint64_t)gridDim.x * blockDim.x) {
    const uint64_t p = parent[c];
    const uint32_t i = inst[c];
    if (p == psk::kEmpty || i >= I) continue;
    if (!psk::main_contains(slots, tdesc[i], p)) atomicOr(err, psk::kErrParentMissing);
  }
}

__global__ void validate_window_kernel(psk::WindowDev w, uint64_t max_blocks, uint32_t* err) {
  for (uint32_t r = blockIdx.x * blockDim.x + threadIdx.x; r < w.R; r += gridDim.x * blockDim.x) {
    const uint64_t a = w.off[r], b = w.off[r + 1];
    const uint32_t L = w.L[r];
    bool ok = b >= a && (b - a) == (uint64_t)(L / 16u) && L < (1u << 30) && b <= max_blocks;
    if (r == 0) ok = ok && a == 0;
    if (!ok) atomicOr(err, psk::kErrWindowLayout);
  }
}

}  // namespace

namespace pskl {

cudaError_t launch_insert_chains(uint64_t* slots, const psk::TableDesc* tdesc, uint32_t I,
                                 unsigned long long* count, uint64_t nchains, const uint32_t* inst,
                                 const uint64_t* off, const uint64_t* hash, uint64_t total,
                                 uint32_t* err, int num_sms, cudaStream_t s) {
  if (total == 0 || nchains == 0) return cudaSuccess;
  uint64_t blocks = (total + 255) / 256;
  const uint64_t cap = (uint64_t)num_sms * 8;
  if (blocks > cap) blocks = cap;
  insert_chains_kernel<<<(unsigned)blocks, 256, 0, s>>>(slots, tdesc, I, count, nchains, inst, off, hash,
                                                        total, err);
  return cudaGetLastError();
}

cudaError_t launch_commit(uint64_t* slots, const psk::TableDesc* tdesc, uint32_t I,
                          unsigned long long* count, const psk::WindowDev& w, const int32_t* assign,
                          const uint32_t* hit_chosen, uint32_t* err, int num_sms, cudaStream_t s) {
  if (w.R == 0) return cudaSuccess;
  uint32_t blocks = (w.R + 7) / 8;
  if (blocks > (uint32_t)num_sms * 8) blocks = num_sms * 8;
  commit_kernel<<<blocks, 256, 0, s>>>(slots, tdesc, I, count, w, assign, hit_chosen, err);
  return cudaGetLastError();
}

cudaError_t launch_check_parents(const uint64_t* slots, const psk::TableDesc* tdesc, uint32_t I,
                                 uint64_t nchains, const uint32_t* inst, const uint64_t* parent,
                                 uint32_t* err, int num_sms, cudaStream_t s) {
  if (nchains == 0) return cudaSuccess;
  uint64_t blocks = (nchains + 255) / 256;
  if (blocks > (uint64_t)num_sms * 8) blocks = (uint64_t)num_sms * 8;
  check_parents_kernel<<<(unsigned)blocks, 256, 0, s>>>(slots, tdesc, I, nchains, inst, parent, err);
  return cudaGetLastError();
}

cudaError_t launch_validate_window(const psk::WindowDev& w, uint64_t max_blocks, uint32_t* err,
                                   cudaStream_t s) {
  if (w.R == 0) return cudaSuccess;
  uint32_t blocks = (w.R + 255) / 256;
  if (blocks > 1024) blocks = 1024;
  validate_window_kernel<<<blocks, 256, 0, s>>>(w, max_blocks, err);
  return cudaGetLastError();
}

}  // namespace pskl
