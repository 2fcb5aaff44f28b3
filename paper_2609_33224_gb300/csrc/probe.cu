// Probe kernel: prefix-hit length of every (request, instance) pair of a window.
//
// hit(r, i) = the first chain position k whose block hash is not cached on instance i (= the
// chain length if every block is cached): the cached prefix of the request on that instance, the
// quantity the paper's scheduler reads from its prefix tree (Section 7) to estimate KVC reuse.
//
// One thread block per request (grid-stride over requests).  The request's chain is staged in
// shared memory once (coalesced 8-byte loads) and reused by every instance's probe; positions past
// the staging capacity are read from global memory (L1/L2-resident: the same block re-reads them).
//   linear mode (any cache): each warp walks one instance at a time, 32 consecutive chain positions
//     per step, __ballot_sync collecting the misses and __ffs finding the first.
//   search mode (prefix-closed caches, where "block k cached" is monotone along the chain): the
//     rows without an earlier prefix in the window come as a list from the relations pass; a work
//     item is (row, chunk of 256 instances), one lane per instance.  A lane first looks up the
//     row's hint position and the one before it together: the hint is the shortest common prefix
//     with the previous requests of the window, which on most instances is exactly the cached
//     prefix (typically a shared system prompt), so most pairs end after one round trip; the
//     others binary-search the rest of their range.
//
// Rows whose chain starts with the whole chain of an earlier request of the window (its base, from
// the relations pass) are derived in a second pass instead: the two chains agree block by block up
// to the base's length nb_b, so on any cache hit(r, i) = hit(base, i) when that is below nb_b, and
// otherwise the first miss lies in [nb_b, nb_r) with everything below known cached.  Only those
// instances (the ones caching the base in full) are searched, by a warp each.  Agentic sessions
// resend their history with each step (Section 3), so most rows of a window are derived.
#include "ps_internal.cuh"

namespace {

constexpr uint32_t kStageBlocks = 4096;  // 32 KB of staged chain per thread block

// Launch statistics (ps_last_probe_stats): each warp adds its threads' counts once, at the end.
enum { kStatRowsScratch = 0, kStatRowsDerived, kStatLookupsScratch, kStatLookupsDerived, kStatChainReads,
       kStatPairsDerived };

__device__ __forceinline__ void add_stat(unsigned long long* p, uint64_t v) {
#pragma unroll
  for (int s = 16; s > 0; s >>= 1) v += __shfl_xor_sync(0xffffffffu, v, s);
  if ((threadIdx.x & 31) == 0 && v) atomicAdd(p, (unsigned long long)v);
}

// Where a pair's result goes: its hit and, when requested, T_pf at that hit (the greedy pass reads
// it instead of recomputing it for pairs whose hit does not change).
struct PairOut {
  uint32_t* hits;
  float* tpf;
  const uint32_t* L;
  psk::DevModel m;
  __device__ __forceinline__ void put(uint32_t r, uint32_t I, uint32_t i, uint32_t h, uint32_t Lr) const {
    hits[(uint64_t)r * I + i] = h;
    if (tpf) tpf[(uint64_t)r * I + i] = psk::t_pf_of_hit(m, Lr, h);
  }
};

template <int WARPS, bool SEARCH>
__global__ void __launch_bounds__(WARPS * 32)
probe_hits_kernel(const uint64_t* __restrict__ slots, const uint64_t* __restrict__ ovf,
                  const psk::TableDesc* __restrict__ tdesc,
                  uint32_t I, const uint64_t* __restrict__ off, const uint64_t* __restrict__ hash,
                  uint32_t R, const psk::RowPre* __restrict__ rows, PairOut out,
                  unsigned long long* __restrict__ stats) {
  extern __shared__ uint64_t s_chain[];
  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  uint64_t n_look = 0, n_rows = 0, n_staged = 0;  // this thread's share of the launch statistics
  for (uint32_t r = blockIdx.x; r < R; r += gridDim.x) {
    if (rows && __ldg(&rows[r].base) >= 0) continue;  // derived in the second pass
    const uint64_t o = off[r];
    const uint64_t nb = off[r + 1] - o;
    const uint32_t Lr = out.tpf ? __ldg(out.L + r) : 0u;
    const uint64_t ns = nb < kStageBlocks ? nb : kStageBlocks;
    if (threadIdx.x == 0) {
      n_rows += 1;
      n_staged += ns;
    }
    for (uint64_t k = threadIdx.x; k < ns; k += WARPS * 32) s_chain[k] = __ldg(hash + o + k);
    __syncthreads();
    auto chain = [&](uint64_t k) { return k < ns ? s_chain[k] : __ldg(hash + o + k); };
    if (SEARCH) {
      for (uint32_t i = threadIdx.x; i < I; i += WARPS * 32) {
        const psk::TableDesc d = tdesc[i];
        uint64_t lo = 0, hi = nb;  // first miss in [lo, hi]
        while (lo < hi) {
          const uint64_t mid = (lo + hi) >> 1;
          ++n_look;
          if (psk::main_contains(slots, ovf, d, chain(mid))) lo = mid + 1; else hi = mid;
        }
        out.put(r, I, i, (uint32_t)lo, Lr);
      }
    } else {
      for (uint32_t i = warp; i < I; i += WARPS) {
        const psk::TableDesc d = tdesc[i];
        auto cached = [&](uint64_t k) {
          ++n_look;
          return psk::main_contains(slots, ovf, d, chain(k));
        };
        const uint64_t h = psk::warp_first_miss_linear(0, nb, cached);
        if (lane == 0) out.put(r, I, i, (uint32_t)h, Lr);
      }
    }
    __syncthreads();
  }
  if (stats) {
    add_stat(stats + kStatRowsScratch, n_rows);
    add_stat(stats + kStatLookupsScratch, n_look);
    add_stat(stats + kStatChainReads, n_staged);
  }
}

// Hint of a row for the search: the shortest common chain prefix with the previous requests of
// the window (0 if there are none).
__device__ __forceinline__ uint32_t row_hint(const psk::RowPre* __restrict__ rows, uint32_t r) {
  uint32_t hint = 0xFFFFFFFFu;
#pragma unroll
  for (int d = 0; d < psk::kLcpBack; ++d)
    if ((uint32_t)d < r) hint = min(hint, __ldg(&rows[r].lcp[d]));
  return hint == 0xFFFFFFFFu ? 0u : hint;
}

// Search mode, rows from the list: see the file comment.
template <int WARPS>
__global__ void __launch_bounds__(WARPS * 32)
probe_search_kernel(const uint64_t* __restrict__ slots, const uint64_t* __restrict__ ovf,
                    const psk::TableDesc* __restrict__ tdesc, uint32_t I, const uint64_t* __restrict__ off,
                    const uint64_t* __restrict__ hash, const psk::RowPre* __restrict__ rows, psk::RowList list,
                    PairOut out, unsigned long long* __restrict__ stats) {
  constexpr uint32_t kChunk = WARPS * 32;
  const uint32_t nchunk = (I + kChunk - 1) / kChunk;
  const uint64_t items = (uint64_t)__ldg(list.count) * nchunk;
  uint64_t n_look = 0, n_rows = 0;
  for (uint64_t item = blockIdx.x; item < items; item += gridDim.x) {
    const uint32_t r = __ldg(list.rows + item / nchunk);
    const uint32_t chunk = (uint32_t)(item % nchunk);
    if (threadIdx.x == 0 && chunk == 0) n_rows += 1;
    const uint32_t i = chunk * kChunk + threadIdx.x;
    if (i >= I) continue;
    const uint64_t o = __ldg(off + r);
    const uint64_t nb = __ldg(off + r + 1) - o;
    const uint64_t* chain = hash + o;
    const psk::TableDesc d = tdesc[i];
    uint64_t lo = 0, hi = nb;  // the first miss lies in [lo, hi]
    if (nb > 0) {
      const uint64_t hint = row_hint(rows, r);
      if (hint == 0 || hint >= nb) {
        const uint64_t p = hint == 0 ? 0 : nb - 1;
        n_look += 1;
        const bool pr = psk::main_contains(slots, ovf, d, __ldg(chain + p));
        if (pr) lo = p + 1; else hi = p;
      } else {
        const uint64_t k1 = __ldg(chain + hint - 1), k2 = __ldg(chain + hint);
        psk::Lookup L1, L2;
        psk::lookup_issue(slots, ovf, d, k1, L1);
        psk::lookup_issue(slots, ovf, d, k2, L2);
        n_look += 2;
        const bool p1 = psk::lookup_finish(slots, ovf, d, k1, L1);
        const bool p2 = psk::lookup_finish(slots, ovf, d, k2, L2);
        if (!p1) hi = hint - 1;
        else if (p2) lo = hint + 1;
        else lo = hi = hint;
      }
    }
    while (lo < hi) {
      const uint64_t mid = (lo + hi) >> 1;
      ++n_look;
      if (psk::main_contains(slots, ovf, d, __ldg(chain + mid))) lo = mid + 1; else hi = mid;
    }
    out.put(r, I, i, (uint32_t)lo, out.tpf ? __ldg(out.L + r) : 0u);
  }
  if (stats) {
    add_stat(stats + kStatRowsScratch, n_rows);
    add_stat(stats + kStatLookupsScratch, n_look);
    add_stat(stats + kStatChainReads, n_look);
  }
}

// Second pass: rows with a base.  One block per row; threads copy the base's hits and collect the
// instances that cache the base in full, then warps search those past the base's end.
template <int WARPS, bool SEARCH>
__global__ void __launch_bounds__(WARPS * 32)
probe_derived_kernel(const uint64_t* __restrict__ slots, const uint64_t* __restrict__ ovf,
                     const psk::TableDesc* __restrict__ tdesc, uint32_t I, const uint64_t* __restrict__ hash,
                     uint32_t R, const psk::RowPre* __restrict__ rows, PairOut out,
                     unsigned long long* __restrict__ stats) {
  extern __shared__ uint32_t s_list[];  // I entries
  __shared__ uint32_t s_n;
  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  uint64_t n_look = 0, n_rows = 0, n_pairs = 0;
  for (uint32_t r = blockIdx.x; r < R; r += gridDim.x) {
    const int32_t b = __ldg(&rows[r].base);
    if (b < 0) continue;  // block-uniform
    if (threadIdx.x == 0) s_n = 0;
    __syncthreads();
    const uint64_t nbb = __ldg(&rows[b].nb);
    const uint64_t nbr = __ldg(&rows[r].nb);
    const uint64_t o = __ldg(&rows[r].off);
    const uint32_t Lr = __ldg(&rows[r].L);
    const uint32_t* hb_row = out.hits + (uint64_t)(uint32_t)b * I;
    for (uint32_t i = threadIdx.x; i < I; i += WARPS * 32) {
      const uint32_t hb = hb_row[i];
      if (hb < nbb || nbb >= nbr) out.put(r, I, i, hb, Lr);
      else s_list[atomicAdd(&s_n, 1u)] = i;
    }
    __syncthreads();
    const uint32_t n = s_n;
    if (threadIdx.x == 0) {
      n_rows += 1;
      n_pairs += n;
    }
    for (uint32_t x = warp; x < n; x += WARPS) {
      const uint32_t i = s_list[x];
      const psk::TableDesc d = tdesc[i];
      auto cached = [&](uint64_t k) {
        ++n_look;
        return psk::main_contains(slots, ovf, d, __ldg(hash + o + k));
      };
      const uint64_t h = SEARCH ? psk::warp_search_range(nbb, nbr, cached) : psk::warp_first_miss_linear(nbb, nbr, cached);
      if (lane == 0) out.put(r, I, i, (uint32_t)h, Lr);
    }
    __syncthreads();
  }
  if (stats) {
    add_stat(stats + kStatRowsDerived, n_rows);
    add_stat(stats + kStatLookupsDerived, n_look);
    add_stat(stats + kStatChainReads, n_look);
    add_stat(stats + kStatPairsDerived, n_pairs);
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
  int per_sm3 = 0;
  cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm3, probe_search_kernel<WARPS>, WARPS * 32, 0);
  if (per_sm3 < per_sm) per_sm = per_sm3;
  if (per_sm < 1) per_sm = 1;
  return per_sm * num_sms;
}

}  // namespace

namespace pskl {

int probe_max_grid(uint32_t I, int num_sms) {
  return I >= 64 ? max_grid<8>(num_sms) : max_grid<4>(num_sms);
}

cudaError_t launch_probe(const uint64_t* slots, const uint64_t* ovf, const psk::TableDesc* tdesc, uint32_t I,
                         const psk::WindowDev& w, const psk::RowPre* rows, psk::RowList list, uint32_t* hits,
                         float* tpf, const psk::DevModel& m, int grid, int search, unsigned long long* stats,
                         cudaEvent_t ev_mid, cudaStream_t s) {
  if (w.R == 0) return cudaSuccess;
  const PairOut out{hits, tpf, w.L, m};
  const int g = (int)((uint32_t)grid < w.R ? (uint32_t)grid : w.R);
  const size_t smem = kStageBlocks * sizeof(uint64_t);
  const size_t smem2 = (size_t)I * sizeof(uint32_t);
#define PS_PROBE(W, S)                                                                                      \
  do {                                                                                                      \
    if (S && rows && list.rows)                                                                             \
      probe_search_kernel<W><<<grid, W * 32, 0, s>>>(slots, ovf, tdesc, I, w.off, w.hash, rows, list, out,   \
                                                     stats);                                                \
    else                                                                                                    \
      probe_hits_kernel<W, S><<<g, W * 32, smem, s>>>(slots, ovf, tdesc, I, w.off, w.hash, w.R, rows, out,  \
                                                     stats);                                                \
    cudaError_t e = cudaGetLastError();                                                                     \
    if (e != cudaSuccess || !rows) return e;                                                                \
    if (ev_mid) cudaEventRecord(ev_mid, s);                                                                 \
    probe_derived_kernel<W, S><<<g, W * 32, smem2, s>>>(slots, ovf, tdesc, I, w.hash, w.R, rows, out,       \
                                                        stats);                                             \
    return cudaGetLastError();                                                                              \
  } while (0)
  if (I >= 64) {
    if (search) PS_PROBE(8, true);
    PS_PROBE(8, false);
  }
  if (search) PS_PROBE(4, true);
  PS_PROBE(4, false);
#undef PS_PROBE
}

}  // namespace pskl
