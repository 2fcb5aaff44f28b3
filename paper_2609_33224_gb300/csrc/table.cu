// Table maintenance kernels: bulk insertion of cached chains, commit of a scheduled window, the
// prefix-closure check and the device-side window layout check.
#include "ps_internal.cuh"

namespace {

// Bulk insert: one warp per instance, the instance's only writer.  The warp scans the chain list
// 32 entries at a time for its own chains and inserts their blocks in order (balanced two-choice
// placement needs the current bucket fill, so each table is written sequentially; different
// instances proceed in parallel).
__global__ void insert_chains_kernel(uint64_t* slots, uint64_t* ovf, const psk::TableDesc* __restrict__ tdesc,
                                     uint32_t I, unsigned long long* count, uint64_t nchains,
                                     const uint32_t* __restrict__ inst, const uint64_t* __restrict__ off,
                                     const uint64_t* __restrict__ hash, uint32_t* err) {
  const int lane = threadIdx.x & 31;
  const uint32_t warps_total = (gridDim.x * blockDim.x) >> 5;
  for (uint32_t i = (blockIdx.x * blockDim.x + threadIdx.x) >> 5; i < I; i += warps_total) {
    const psk::TableDesc d = tdesc[i];
    unsigned long long added = 0;
    bool full = false, reserved = false;
    for (uint64_t c0 = 0; c0 < nchains; c0 += 32) {
      const uint64_t c = c0 + lane;
      unsigned mine = __ballot_sync(0xffffffffu, c < nchains && __ldg(inst + c) == i);
      while (mine) {
        const int l = __ffs(mine) - 1;
        mine &= mine - 1;
        const uint64_t a = __ldg(off + c0 + l), b = __ldg(off + c0 + l + 1);
        for (uint64_t k = a; k < b && !full; ++k) {
          const uint64_t key = __ldg(hash + k);
          if (key == psk::kEmpty || key == psk::kTomb) {
            reserved = true;
            continue;
          }
          const int res = psk::warp_insert(slots, ovf, d, key);
          if (res > 0) ++added;
          if (res < 0) full = true;
        }
      }
    }
    if (lane == 0) {
      count[i] += added;
      if (full) atomicOr(err, psk::kErrTableFull);
      if (reserved) atomicOr(err, psk::kErrReservedHash);
    }
  }
}

// Instance ids must be valid before the per-instance scan (a chain with a bad id is never seen).
__global__ void check_instances_kernel(uint32_t I, uint64_t nchains, const uint32_t* __restrict__ inst,
                                       uint32_t* err) {
  for (uint64_t c = blockIdx.x * (uint64_t)blockDim.x + threadIdx.x; c < nchains; c += (uint64_t)gridDim.x * blockDim.x)
    if (inst[c] >= I) atomicOr(err, psk::kErrBadInstance);
}

// Commit: each admitted request caches its uncached blocks chain[h..nb) on its instance; one warp
// per instance applies that instance's requests in arrival order.
__global__ void commit_kernel(uint64_t* slots, uint64_t* ovf, const psk::TableDesc* __restrict__ tdesc, uint32_t I,
                              unsigned long long* count, psk::WindowDev w, const int32_t* __restrict__ assign,
                              const uint32_t* __restrict__ hit_chosen, uint32_t* err) {
  const int lane = threadIdx.x & 31;
  const uint32_t warps_total = (gridDim.x * blockDim.x) >> 5;
  for (uint32_t i = (blockIdx.x * blockDim.x + threadIdx.x) >> 5; i < I; i += warps_total) {
    const psk::TableDesc d = tdesc[i];
    unsigned long long added = 0;
    bool full = false;
    for (uint32_t r0 = 0; r0 < w.R; r0 += 32) {
      const uint32_t r = r0 + lane;
      unsigned mine = __ballot_sync(0xffffffffu, r < w.R && assign[r] == (int32_t)i);
      while (mine) {
        const int l = __ffs(mine) - 1;
        mine &= mine - 1;
        const uint64_t o = w.off[r0 + l];
        const uint64_t nb = w.off[r0 + l + 1] - o;
        for (uint64_t k = hit_chosen[r0 + l]; k < nb && !full; ++k) {
          const uint64_t key = w.hash[o + k];
          if (key == psk::kEmpty || key == psk::kTomb) continue;
          const int res = psk::warp_insert(slots, ovf, d, key);
          if (res > 0) ++added;
          if (res < 0) full = true;
        }
      }
    }
    if (lane == 0) {
      count[i] += added;
      if (full) atomicOr(err, psk::kErrTableFull);
    }
  }
}

// Prefix closure check (search mode): every chain's parent must be cached once the chains are in.
__global__ void check_parents_kernel(const uint64_t* slots, const uint64_t* ovf, const psk::TableDesc* __restrict__ tdesc, uint32_t I,
                                     uint64_t nchains, const uint32_t* __restrict__ inst,
                                     const uint64_t* __restrict__ parent, uint32_t* err) {
  for (uint64_t c = blockIdx.x * (uint64_t)blockDim.x + threadIdx.x; c < nchains; c += (uint64_t)gridDim.x * blockDim.x) {
    const uint64_t p = parent[c];
    const uint32_t i = inst[c];
    if (p == psk::kEmpty || i >= I) continue;
    if (!psk::main_contains(slots, ovf, tdesc[i], p)) atomicOr(err, psk::kErrParentMissing);
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

cudaError_t launch_insert_chains(uint64_t* slots, uint64_t* ovf, const psk::TableDesc* tdesc, uint32_t I,
                                 unsigned long long* count, uint64_t nchains, const uint32_t* inst,
                                 const uint64_t* off, const uint64_t* hash, uint64_t total,
                                 uint32_t* err, int num_sms, cudaStream_t s) {
  if (total == 0 || nchains == 0) return cudaSuccess;
  uint64_t blocks = (nchains + 255) / 256;
  if (blocks > (uint64_t)num_sms * 8) blocks = (uint64_t)num_sms * 8;
  check_instances_kernel<<<(unsigned)blocks, 256, 0, s>>>(I, nchains, inst, err);
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  const uint32_t warps_per_block = 4;
  insert_chains_kernel<<<(I + warps_per_block - 1) / warps_per_block, 32 * warps_per_block, 0, s>>>(
      slots, ovf, tdesc, I, count, nchains, inst, off, hash, err);
  return cudaGetLastError();
}

cudaError_t launch_commit(uint64_t* slots, uint64_t* ovf, const psk::TableDesc* tdesc, uint32_t I,
                          unsigned long long* count, const psk::WindowDev& w, const int32_t* assign,
                          const uint32_t* hit_chosen, uint32_t* err, int num_sms, cudaStream_t s) {
  (void)num_sms;
  if (w.R == 0) return cudaSuccess;
  const uint32_t warps_per_block = 4;
  commit_kernel<<<(I + warps_per_block - 1) / warps_per_block, 32 * warps_per_block, 0, s>>>(
      slots, ovf, tdesc, I, count, w, assign, hit_chosen, err);
  return cudaGetLastError();
}

cudaError_t launch_check_parents(const uint64_t* slots, const uint64_t* ovf, const psk::TableDesc* tdesc, uint32_t I,
                                 uint64_t nchains, const uint32_t* inst, const uint64_t* parent,
                                 uint32_t* err, int num_sms, cudaStream_t s) {
  if (nchains == 0) return cudaSuccess;
  uint64_t blocks = (nchains + 255) / 256;
  if (blocks > (uint64_t)num_sms * 8) blocks = (uint64_t)num_sms * 8;
  check_parents_kernel<<<(unsigned)blocks, 256, 0, s>>>(slots, ovf, tdesc, I, nchains, inst, parent, err);
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
