// Fused score kernel: hit lengths + instance state -> predicted latencies, Algorithm 1's admission
// sets and the per-request pick, each request independently against the same state.
//
// One warp per request (grid-stride).  Lane l handles instances l, l+32, ...  Pass 1 evaluates the
// capacity guard and the recompute cost W (Alg. 1 KVC-first filtering) and reduces W_min over A with
// warp shuffles; pass 2 classifies each pair (Eq. 8 filter, TPOT and TTFT admission), writes the
// optional per-pair outputs, and reduces the lexicographic (class, value, instance) key to the
// pick: D-C-Q inside T, the LMetric product inside C when T is empty, Reject when A is empty.
#include "ps_internal.cuh"

namespace {

__global__ void __launch_bounds__(256)
score_rows_kernel(const uint32_t* __restrict__ hits, psk::StateSoA st, uint32_t I, psk::WindowDev w,
                  psk::DevModel m, float* __restrict__ tpot_out, float* __restrict__ ttft_out,
                  uint8_t* __restrict__ cls_out, int32_t* __restrict__ best_out,
                  uint8_t* __restrict__ path_out) {
  const int lane = threadIdx.x & 31;
  const uint32_t warps_total = (gridDim.x * blockDim.x) >> 5;
  for (uint32_t r = (blockIdx.x * blockDim.x + threadIdx.x) >> 5; r < w.R; r += warps_total) {
    const psk::RowConst rc = psk::row_const(m, w.L[r], w.ttft_t[r], w.tpot_t[r]);
    const uint32_t* hrow = hits + (uint64_t)r * I;
    float wmin = INFINITY;
    bool anyA = false;
    for (uint32_t i = lane; i < I; i += 32) {
      const psk::PairEval e = psk::eval_pair(m, rc, __ldg(hrow + i), __ldg(st.b + i), __ldg(st.qr + i),
                                             __ldg(st.q + i), __ldg(st.S + i), __ldg(st.M + i),
                                             __ldg(st.Bmax + i));
      if (e.inA) {
        wmin = fminf(wmin, e.W);
        anyA = true;
      }
    }
    anyA = __any_sync(0xffffffffu, anyA);
    wmin = psk::warp_fmin(wmin);
    psk::ArgKey best{psk::kNoKeyCi, ~0ull};
    for (uint32_t i = lane; i < I; i += 32) {
      const uint32_t h = __ldg(hrow + i);
      const int32_t b = __ldg(st.b + i), qr = __ldg(st.qr + i);
      const int64_t q = __ldg(st.q + i);
      const psk::PairEval e = psk::eval_pair(m, rc, h, b, qr, q, __ldg(st.S + i), __ldg(st.M + i),
                                             __ldg(st.Bmax + i));
      const uint32_t cls = e.inA ? psk::pair_class(m, rc, e, wmin) : 3u;
      const uint64_t x = (uint64_t)r * I + i;
      if (tpot_out) tpot_out[x] = e.tpot;
      if (ttft_out) ttft_out[x] = e.ttft;
      if (cls_out) cls_out[x] = (uint8_t)cls;
      if (cls <= 1u) {
        const psk::ArgKey k{(cls << 28) | i, psk::pair_value(cls, h, b, qr, q, e.n)};
        if (psk::key_less(k, best)) best = k;
      }
    }
    best = psk::warp_argmin(best);
    if (lane == 0) {
      const bool pick = anyA && best.ci != psk::kNoKeyCi;
      if (best_out) best_out[r] = pick ? (int32_t)(best.ci & 0x0FFFFFFFu) : -1;
      if (path_out) path_out[r] = pick ? (uint8_t)(best.ci >> 28) : (uint8_t)2;
    }
  }
}

}  // namespace

namespace pskl {

cudaError_t launch_score(const uint32_t* hits, psk::StateSoA st, uint32_t I, const psk::WindowDev& w,
                         const psk::DevModel& m, float* tpot, float* ttft, uint8_t* cls, int32_t* best,
                         uint8_t* path, int num_sms, cudaStream_t s) {
  if (w.R == 0) return cudaSuccess;
  const uint32_t rows_per_block = 8;
  uint32_t grid = (w.R + rows_per_block - 1) / rows_per_block;
  const uint32_t cap = (uint32_t)num_sms * 8u;
  if (grid > cap) grid = cap;
  score_rows_kernel<<<grid, 256, 0, s>>>(hits, st, I, w, m, tpot, ttft, cls, best, path);
  return cudaGetLastError();
}

}  // namespace pskl
