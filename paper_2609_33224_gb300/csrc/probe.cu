// Probe kernel: prefix-hit length of every (request, instance) pair of a window.
//
// hit(r, i) = the first chain position k whose block hash is not cached on instance i (= the
// chain length if every block is cached): the cached prefix of the request on that instance, the
// quantity the paper's scheduler reads from its prefix tree (Section 6) to estimate KVC reuse.
//
// One thread block per request (grid-stride over requests).  The request's chain is staged in
// shared memory once (coalesced 8-byte loads) and reused by every instance's walk.  Each warp
// handles one instance at a time with 32 probes per step, __ballot_sync collecting the misses and
// __ffs finding the first: either a linear walk over 32 consecutive positions per step, or (for
// prefix-closed caches) a 32-ary search over 32 evenly spaced positions.  Positions past the staging
// capacity are read from global memory (L1/L2-resident: the same block re-reads them).
#include "ps_internal.cuh"

namespace {

constexpr uint32_t kStageBlocks = 8192;  // 64 KB of staged chain per thread block

template <int WARPS, bool SEARCH>
__global__ void __launch_bounds__(WARPS * 32)
probe_hits_kernel(const uint64_t* __restrict__ slots, const uint64_t* __restrict__ ovf,
                  const psk::TableDesc* __restrict__ tdesc,
                  uint32_t I, const uint64_t* __restrict__ off, const uint64_t* __restrict__ hash,
                  uint32_t R, uint32_t* __restrict__ hits) {
  extern __shared__ uint64_t s_chain[];
  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  for (uint32_t r = blockIdx.x; r < R; r += gridDim.x) {
    const uint64_t o = off[r];
    const uint64_t nb = off[r + 1] - o;
    const uint64_t ns = nb < kStageBlocks ? nb : kStageBlocks;
    for (uint64_t k = threadIdx.x; k < ns; k += WARPS * 32) s_chain[k] = __ldg(hash + o + k);
    __syncthreads();
    for (uint32_t i = warp; i < I; i += WARPS) {
      const psk::TableDesc d = tdesc[i];
      auto cached = [&](uint64_t k) {
        const uint64_t key = k < ns ? s_chain[k] : __ldg(hash + o + k);
        return psk::main_contains(slots, ovf, d, key);
      };
      const uint64_t h = SEARCH ? psk::warp_first_miss_search(0, nb, cached)
                                : psk::warp_first_miss_linear(0, nb, cached);
      if (lane == 0) hits[(uint64_t)r * I + i] = (uint32_t)h;
    }
    __syncthreads();
  }
}

template <int WARPS>
int max_grid(int num_sms) {
  int per_sm = 0, per_sm2 = 0;
  const int smem = (int)(kStageBlocks * sizeof(uint64_t));
  cudaFuncSetAttribute(probe_hits_kernel<WARPS, false>, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
  cudaFuncSetAttribute(probe_hits_kernel<WARPS, true>, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
  cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, probe_hits_kernel<WARPS, false>, WARPS * 32, smem);
  cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm2, probe_hits_kernel<WARPS, true>, WARPS * 32, smem);
  if (per_sm2 < per_sm) per_sm = per_sm2;
  if (per_sm < 1) per_sm = 1;
  return per_sm * num_sms;
}

}  // namespace

namespace pskl {

int probe_max_grid(uint32_t I, int num_sms) {
  return I >= 64 ? max_grid<16>(num_sms) : max_grid<4>(num_sms);
}

cudaError_t launch_probe(const uint64_t* slots, const uint64_t* ovf, const psk::TableDesc* tdesc, uint32_t I,
                         const psk::WindowDev& w, uint32_t* hits, int grid, int search, cudaStream_t s) {
  if (w.R == 0) return cudaSuccess;
  const int g = (int)((uint32_t)grid < w.R ? (uint32_t)grid : w.R);
  const size_t smem = kStageBlocks * sizeof(uint64_t);
  if (I >= 64) {
    if (search)
      probe_hits_kernel<16, true><<<g, 16 * 32, smem, s>>>(slots, ovf, tdesc, I, w.off, w.hash, w.R, hits);
    else
      probe_hits_kernel<16, false><<<g, 16 * 32, smem, s>>>(slots, ovf, tdesc, I, w.off, w.hash, w.R, hits);
  } else {
    if (search)
      probe_hits_kernel<4, true><<<g, 4 * 32, smem, s>>>(slots, ovf, tdesc, I, w.off, w.hash, w.R, hits);
    else
      probe_hits_kernel<4, false><<<g, 4 * 32, smem, s>>>(slots, ovf, tdesc, I, w.off, w.hash, w.R, hits);
  }
  return cudaGetLastError();
}

}  // namespace pskl
