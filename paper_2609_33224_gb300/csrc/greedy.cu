// Greedy in-window assignment (Algorithm 1 applied to the window's requests in arrival order).
//
// The paper's gateway decides each request online and updates the instance records along the
// request path before the next decision (Section 4, Metadata service; Section 6).  This kernel
// replays that sequence for a whole window on the GPU: one persistent thread block whose threads
// each own up to IPT instances.  Per request r:
//   1. hit of r on instance i = hit0[r][i] (the probe kernel's result on the committed tables)
//      extended through the window's delta table: an instance that has received blocks in this
//      window is re-probed at position hit0, and if that block is now cached a warp finds the new
//      first miss over delta and main (linear walk, or 32-ary search on prefix-closed caches: the
//      delta only ever adds a chain's continuation to a cached prefix, so closure is kept).
//      Instances untouched in the window need no probe.
//   2. the whole row is re-evaluated from the current state (capacity guard, W, W_min, Eq. 8
//      filter, TPOT/TTFT admission, D-C-Q key or LMetric fallback), reduced block-wide to the pick;
//   3. the pick's state is updated (qr += 1, q += n, S += L) and its uncached blocks
//      chain[h..nb) are inserted into the delta table for instance j.
// The next request's row constants, hit row and the chain blocks at its hit positions are loaded
// while the current request is decided, so a step starts with its inputs in registers.
// Committed tables are never written here; the decisions and the updated state are a pending
// window that ps_commit_window applies.  No step waits on another block: a single thread block with
// __syncthreads barriers only.
#include "ps_internal.cuh"

namespace {

struct RowIn {
  uint64_t o, nb;
  uint32_t L;
  float ttft_t, tpot_t;
};

__device__ __forceinline__ RowIn load_row(const psk::WindowDev& w, uint32_t r) {
  RowIn x;
  x.o = w.off[r];
  x.nb = w.off[r + 1] - x.o;
  x.L = w.L[r];
  x.ttft_t = w.ttft_t[r];
  x.tpot_t = w.tpot_t[r];
  return x;
}

// Block-wide reductions without an extra barrier: after the per-warp partials are in shared
// memory (and one __syncthreads), every warp reduces the (up to 32) partials with shuffles.
__device__ __forceinline__ void cross_warp_min_any(const float* s_w, const int* s_a, int nw, float& wmin,
                                                   bool& anyA) {
  const int lane = threadIdx.x & 31;
  const float v = lane < nw ? s_w[lane] : INFINITY;
  const bool a = lane < nw ? (s_a[lane] != 0) : false;
  wmin = psk::warp_fmin(v);
  anyA = __any_sync(0xffffffffu, a);
}

__device__ __forceinline__ psk::ArgKey cross_warp_argmin(const psk::ArgKey* s_k, int nw) {
  const int lane = threadIdx.x & 31;
  psk::ArgKey k = lane < nw ? s_k[lane] : psk::ArgKey{psk::kNoKeyCi, ~0ull};
  return psk::warp_argmin(k);
}

template <int IPT, bool SEARCH>
__global__ void __launch_bounds__(1024, 1)
greedy_kernel(const uint64_t* __restrict__ slots, const uint64_t* __restrict__ ovf,
              const psk::TableDesc* __restrict__ tdesc, uint32_t I,
              psk::WindowDev w, const uint32_t* __restrict__ hit0, psk::StateSoA committed,
              psk::StateSoA pending, psk::DevModel m, psk::DeltaSlot* delta, uint32_t delta_nbkt,
              int32_t* __restrict__ assign, uint8_t* __restrict__ path, uint32_t* __restrict__ hit_chosen,
              uint32_t* err) {
  extern __shared__ unsigned long long smem_raw[];
  int64_t* s_q = reinterpret_cast<int64_t*>(smem_raw);
  int64_t* s_S = s_q + I;
  int64_t* s_M = s_S + I;
  int32_t* s_b = reinterpret_cast<int32_t*>(s_M + I);
  int32_t* s_qr = s_b + I;
  int32_t* s_Bmax = s_qr + I;
  uint32_t* s_h = reinterpret_cast<uint32_t*>(s_Bmax + I);
  uint32_t* s_walk = s_h + I;
  uint32_t* s_end = s_walk + I;  // chain end of the last request assigned to the instance this window
  psk::InstTerms* s_it = reinterpret_cast<psk::InstTerms*>(s_end + I);
  uint8_t* s_touched = reinterpret_cast<uint8_t*>(s_it + I);
  __shared__ float s_red_w[32];
  __shared__ int s_red_a[32];
  __shared__ psk::ArgKey s_red_k[32];
  __shared__ uint32_t s_nwalk;

  const int t = threadIdx.x;
  const int NT = blockDim.x;
  const int lane = t & 31;
  const int warp = t >> 5;
  const int NW = NT >> 5;

  for (uint32_t i = t; i < I; i += NT) {
    s_b[i] = committed.b[i];
    s_qr[i] = committed.qr[i];
    s_q[i] = committed.q[i];
    s_S[i] = committed.S[i];
    s_M[i] = committed.M[i];
    s_Bmax[i] = committed.Bmax[i];
    s_end[i] = 0;
    s_touched[i] = 0;
    s_it[i] = psk::inst_terms(m, s_b[i], s_qr[i], s_q[i], s_Bmax[i]);
  }
  if (t == 0) s_nwalk = 0;
  // Inputs of the next request: row constants, hit row, chain block at each hit position.
  RowIn nx{};
  uint32_t hn[IPT];
  uint64_t cn[IPT];
  if (w.R > 0) nx = load_row(w, 0);
#pragma unroll
  for (int k = 0; k < IPT; ++k) {
    const uint32_t i = t + k * NT;
    hn[k] = (i < I && w.R > 0) ? __ldg(hit0 + i) : 0u;
    cn[k] = (i < I && hn[k] < nx.nb) ? w.hash[nx.o + hn[k]] : 0ull;
  }
  __syncthreads();

  for (uint32_t r = 0; r < w.R; ++r) {
    const RowIn cur = nx;
    const uint64_t o = cur.o;
    const uint64_t nb = cur.nb;
    const psk::RowConst rc = psk::row_const(m, cur.L, cur.ttft_t, cur.tpot_t);
    uint32_t hc[IPT];
#pragma unroll
    for (int k = 0; k < IPT; ++k) {
      const uint32_t i = t + k * NT;
      hc[k] = hn[k];
      if (i < I) {
        if (s_touched[i] && hc[k] < nb && psk::delta_contains(delta, delta_nbkt, i, cn[k])) {
          const uint32_t at = atomicAdd(&s_nwalk, 1u);
          s_walk[at] = i;
        }
        s_h[i] = hc[k];
      }
    }
    // first half of the prefetch: row constants and hit row of request r + 1
    const bool more = r + 1 < w.R;
    if (more) {
      nx = load_row(w, r + 1);
#pragma unroll
      for (int k = 0; k < IPT; ++k) {
        const uint32_t i = t + k * NT;
        if (i < I) hn[k] = __ldg(hit0 + (uint64_t)(r + 1) * I + i);
      }
    }
    __syncthreads();  // (A) hits staged, walk list complete
    const uint32_t nwalk = s_nwalk;
    if (nwalk) {
      for (uint32_t x = warp; x < nwalk; x += NW) {
        const uint32_t i = s_walk[x];
        const psk::TableDesc d = tdesc[i];
        // Positions past hit0 are never in a prefix-closed main table (hit0 is its first miss), so
        // the search only consults the delta; the linear walk checks both.
        auto cached = [&](uint64_t k) {
          const uint64_t key = w.hash[o + k];
          return psk::delta_contains(delta, delta_nbkt, i, key) ||
                 (!SEARCH && psk::main_contains(slots, ovf, d, key));
        };
        // Likely answer: where the last request assigned to i in this window ended (the same
        // session's previous step usually ends exactly there).
        const uint64_t from = (uint64_t)s_h[i] + 1;
        const uint64_t hnew = SEARCH ? psk::warp_first_miss_search_hint(from, nb, s_end[i], cached)
                                     : psk::warp_first_miss_linear(from, nb, cached);
        if (lane == 0) s_h[i] = (uint32_t)hnew;
      }
      __syncthreads();  // (B) extended hits visible
#pragma unroll
      for (int k = 0; k < IPT; ++k) {
        const uint32_t i = t + k * NT;
        if (i < I) hc[k] = s_h[i];
      }
    }
    // Pass 1: capacity guard and recompute cost; W_min over A.
    psk::PairEval ev[IPT];
    float wmin = INFINITY;
    bool anyA = false;
#pragma unroll
    for (int k = 0; k < IPT; ++k) {
      const uint32_t i = t + k * NT;
      if (i < I) {
        ev[k] = psk::eval_pair_terms(m, rc, hc[k], s_it[i], s_q[i], s_S[i], s_M[i]);
        if (ev[k].inA) {
          wmin = fminf(wmin, ev[k].W);
          anyA = true;
        }
      } else {
        ev[k].inA = false;
      }
    }
    wmin = psk::warp_fmin(wmin);
    anyA = __any_sync(0xffffffffu, anyA);
    if (lane == 0) {
      s_red_w[warp] = wmin;
      s_red_a[warp] = anyA ? 1 : 0;
    }
    __syncthreads();  // (C)
    cross_warp_min_any(s_red_w, s_red_a, NW, wmin, anyA);
    // second half of the prefetch: chain blocks of request r + 1 at its hit positions
    if (more) {
#pragma unroll
      for (int k = 0; k < IPT; ++k) {
        const uint32_t i = t + k * NT;
        if (i < I && hn[k] < nx.nb) cn[k] = w.hash[nx.o + hn[k]];
      }
    }
    // Pass 2: admission classes and the lexicographic argmin.
    psk::ArgKey best{psk::kNoKeyCi, ~0ull};
#pragma unroll
    for (int k = 0; k < IPT; ++k) {
      const uint32_t i = t + k * NT;
      if (i < I && ev[k].inA) {
        const uint32_t cls = psk::pair_class(m, rc, ev[k], wmin);
        if (cls <= 1u) {
          const psk::ArgKey kk{(cls << 28) | i, psk::pair_value(cls, hc[k], s_b[i], s_qr[i], s_q[i], ev[k].n)};
          if (psk::key_less(kk, best)) best = kk;
        }
      }
    }
    best = psk::warp_argmin(best);
    if (lane == 0) s_red_k[warp] = best;
    __syncthreads();  // (D)
    best = cross_warp_argmin(s_red_k, NW);
    const bool pick = anyA && best.ci != psk::kNoKeyCi;
    const uint32_t j = best.ci & 0x0FFFFFFFu;
    const uint32_t hj = pick ? s_h[j] : 0u;
    if (t == 0) {
      assign[r] = pick ? (int32_t)j : -1;
      path[r] = pick ? (uint8_t)(best.ci >> 28) : (uint8_t)2;
      hit_chosen[r] = hj;
      if (pick) {
        s_qr[j] += 1;
        s_q[j] += (int64_t)rc.L - 16 * (int64_t)hj;
        s_S[j] += (int64_t)rc.L;
        s_end[j] = (uint32_t)nb;
        s_touched[j] = 1;
        s_it[j] = psk::inst_terms(m, s_b[j], s_qr[j], s_q[j], s_Bmax[j]);
      }
      s_nwalk = 0;
    }
    if (pick) {
      for (uint64_t k = (uint64_t)hj + t; k < nb; k += NT)
        if (!psk::delta_insert(delta, delta_nbkt, j, w.hash[o + k])) atomicOr(err, psk::kErrDeltaFull);
    }
    __syncthreads();  // (E) state, delta and walk counter ready for the next request
  }
  for (uint32_t i = t; i < I; i += NT) {
    pending.b[i] = s_b[i];
    pending.qr[i] = s_qr[i];
    pending.q[i] = s_q[i];
    pending.S[i] = s_S[i];
    pending.M[i] = s_M[i];
    pending.Bmax[i] = s_Bmax[i];
  }
}

size_t greedy_smem(uint32_t I) {
  return (size_t)I * (3 * sizeof(int64_t) + 3 * sizeof(int32_t) + 3 * sizeof(uint32_t) + sizeof(psk::InstTerms) + 1) + 16;
}

template <int IPT, bool SEARCH>
cudaError_t greedy_launch(const uint64_t* slots, const uint64_t* ovf, const psk::TableDesc* tdesc, uint32_t I,
                          const psk::WindowDev& w, const uint32_t* hit0, psk::StateSoA committed,
                          psk::StateSoA pending, const psk::DevModel& m, psk::DeltaSlot* delta,
                          uint32_t delta_nbkt, int32_t* assign, uint8_t* path, uint32_t* hit_chosen,
                          uint32_t* err, uint32_t nt, cudaStream_t s) {
  const size_t smem = greedy_smem(I);
  cudaError_t e = cudaFuncSetAttribute(greedy_kernel<IPT, SEARCH>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       (int)smem);
  if (e != cudaSuccess) return e;
  greedy_kernel<IPT, SEARCH><<<1, nt, smem, s>>>(slots, ovf, tdesc, I, w, hit0, committed, pending, m, delta,
                                                 delta_nbkt, assign, path, hit_chosen, err);
  return cudaGetLastError();
}

}  // namespace

namespace pskl {

cudaError_t launch_greedy(const uint64_t* slots, const uint64_t* ovf, const psk::TableDesc* tdesc, uint32_t I,
                          const psk::WindowDev& w, const uint32_t* hit0, psk::StateSoA committed,
                          psk::StateSoA pending, const psk::DevModel& m, psk::DeltaSlot* delta,
                          uint32_t delta_nbkt, int32_t* assign, uint8_t* path, uint32_t* hit_chosen,
                          uint32_t* err, int search, cudaStream_t s) {
  uint32_t nt = (I + 31) / 32 * 32;
  if (nt > 1024) nt = 1024;
  const uint32_t ipt = (I + nt - 1) / nt;
#define PS_GREEDY(IPT)                                                                                         \
  return search ? greedy_launch<IPT, true>(slots, ovf, tdesc, I, w, hit0, committed, pending, m, delta,        \
                                           delta_nbkt, assign, path, hit_chosen, err, nt, s)                   \
                : greedy_launch<IPT, false>(slots, ovf, tdesc, I, w, hit0, committed, pending, m, delta,       \
                                            delta_nbkt, assign, path, hit_chosen, err, nt, s)
  if (ipt <= 1) PS_GREEDY(1);
  if (ipt <= 2) PS_GREEDY(2);
  if (ipt <= 4) PS_GREEDY(4);
#undef PS_GREEDY
  return cudaErrorInvalidValue;
}

// The delta table only holds one window's blocks: clear it whole after each window.
cudaError_t launch_delta_clear(psk::DeltaSlot* delta, uint64_t nslots, cudaStream_t s) {
  return cudaMemsetAsync(delta, 0, nslots * sizeof(psk::DeltaSlot), s);
}

}  // namespace pskl
