// Window staging in the shared-prefix form (ps_window.parent): every request's chain rebuilt on the
// device from its ancestors' own blocks.
//
// An agentic session resends its history with every step (Section 3), so most requests of a window
// extend an earlier request's prompt.  In the shared-prefix form the host sends each request's own
// blocks only, with a parent link: request r's chain is its parent's whole chain followed by r's own
// blocks.  Ancestor a of r (r itself included) owns the chain positions [nb(parent(a)), nb(a)), so
// r's chain is the concatenation of its ancestors' own blocks, root first.  One warp per request walks
// its parent links and copies each ancestor's blocks into place (coalesced); every position of every
// chain is written once.
#include "ps_internal.cuh"

namespace {

__global__ void __launch_bounds__(256)
expand_chains_kernel(const uint64_t* __restrict__ full_off, const uint64_t* __restrict__ own_off,
                     const uint64_t* __restrict__ own_hash, const int32_t* __restrict__ parent, uint32_t R,
                     uint64_t* __restrict__ hash, uint32_t* err) {
  const int lane = threadIdx.x & 31;
  const uint32_t warps = (gridDim.x * blockDim.x) >> 5;
  for (uint32_t r = (blockIdx.x * blockDim.x + threadIdx.x) >> 5; r < R; r += warps) {
    const uint64_t base = __ldg(full_off + r);
    int32_t a = (int32_t)r;
    uint32_t steps = 0;
    while (a >= 0) {
      const uint64_t a_off = __ldg(own_off + a);
      const uint64_t a_n = __ldg(own_off + a + 1) - a_off;
      const int32_t p = __ldg(parent + a);
      const uint64_t start = p >= 0 ? __ldg(full_off + p + 1) - __ldg(full_off + p) : 0ull;  // first position a owns
      for (uint64_t k = (uint64_t)lane; k < a_n; k += 32) hash[base + start + k] = __ldg(own_hash + a_off + k);
      // parents precede their children (checked on the host), so the walk ends within r steps
      if (++steps > r + 1u) {
        if (lane == 0) atomicOr(err, psk::kErrWindowLayout);
        break;
      }
      a = p;
    }
  }
}

}  // namespace

namespace pskl {

cudaError_t launch_expand_chains(const uint64_t* full_off, const uint64_t* own_off, const uint64_t* own_hash,
                                 const int32_t* parent, uint32_t R, uint64_t* hash, uint32_t* err, int num_sms,
                                 cudaStream_t s) {
  if (R == 0) return cudaSuccess;
  uint32_t grid = (R + 7u) / 8u;  // 8 warps (requests) per block
  const uint32_t cap = (uint32_t)num_sms * 8u;
  if (grid > cap) grid = cap;
  expand_chains_kernel<<<grid, 256, 0, s>>>(full_off, own_off, own_hash, parent, R, hash, err);
  return cudaGetLastError();
}

}  // namespace pskl
