// Probe kernel: prefix-hit length of every (request, instance) pair of a window.
//
// hit(r, i) = the first chain position k whose block hash is not cached on instance i (= the
// chain length if every block is cached): the cached prefix of the request on that instance, the
// quantity the paper's scheduler reads from its prefix tree (Section 6) to estimate KVC reuse.
//
// One thread block per request (grid-stride over requests).  The request's chain is staged in
// shared memory once (coalesced 8-byte loads) and reused by every instance's walk.  Each warp walks
// one instance at a time, 32 chain positions per step: lane k probes position base + k in the
// instance's table, __ballot_sync collects the misses and __ffs finds the first.  Positions past the
// staging capacity are read from global memory (L1/L2-resident: the same block re-reads them).
#include "ps_internal.cuh"

namespace {

constexpr uint32_t kStageBlocks = 8192;  // 64 KB of staged chain per thread block

template <int WARPS>
__global__ void __launch_bounds__(WARPS * 32)
probe_hits_kernel(const uint64_t* __restrict__ slots, const psk::TableDesc* __restrict__ tdesc,
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
      uint64_t h = nb;
      for (uint64_t base = 0; base < nb; base += 32) {
        const uint64_t k = base + lane;
        bool present = true;  // positions past the chain end never count as a miss
        if (k < nb) {
          const uint64_t key = k < ns ? s_chain[k] : __ldg(hash + o + k);
          present = psk::main_contains(slots, d, key);
        }
        const unsigned miss = __ballot_sync(0xffffffffu, !present);
        if (miss) {
          h = base + (uint64_t)(__ffs(miss) - 1);
          break;
        }
      }
      if (lane == 0) hits[(uint64_t)r * I + i] = (uint32_t)h;
    }
    __syncthreads();
  }
}

template <int WARPS>
int max_grid(int num_sms) {
  int per_sm = 0;
  cudaFuncSetAttribute(probe_hits_kernel<WARPS>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                       (int)(kStageBlocks * sizeof(uint64_t)));
  cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, probe_hits_kernel<WARPS>, WARPS * 32,
                                                kStageBlocks * sizeof(uint64_t));
  if (per_sm < 1) per_sm = 1;
  return per_sm * num_sms;
}

}  // namespace

namespace pskl {

int probe_max_grid(uint32_t I, int num_sms) {
  return I >= 64 ? max_grid<16>(num_sms) : max_grid<4>(num_sms);
}

cudaError_t launch_probe(const uint64_t* slots, const psk::TableDesc* tdesc, uint32_t I,
                         const psk::WindowDev& w, uint32_t* hits, int grid, cudaStream_t s) {
  if (w.R == 0) return cudaSuccess;
  const int g = (int)((uint32_t)grid < w.R ? (uint32_t)grid : w.R);
  const size_t smem = kStageBlocks * sizeof(uint64_t);
  if (I >= 64)
    probe_hits_kernel<16><<<g, 16 * 32, smem, s>>>(slots, tdesc, I, w.off, w.hash, w.R, hits);
  else
    probe_hits_kernel<4><<<g, 4 * 32, smem, s>>>(slots, tdesc, I, w.off, w.hash, w.R, hits);
  return cudaGetLastError();
}

}  // namespace pskl
