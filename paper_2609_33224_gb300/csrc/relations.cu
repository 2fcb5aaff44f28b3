// Per-request window constants for the greedy pass, computed for all requests in parallel.
//
// Besides the Algorithm 1 / Eq. 8 row constants (T_pf(0, L), CacheBenefit Z, eta * Z, the TTFT
// budget), each request gets its chain relations to earlier requests of the same window:
//   * lcp[d - 1]: the common chain prefix with the request d places before it (d = 1..kLcpBack).  Chained
//     block hashes (Section 7's prefix tree) make "block k equal" imply "blocks 0..k equal", so the
//     common prefix is found with the 32-ary first-miss search.
//   * par: the deepest earlier request whose whole chain is a prefix of this one (an agentic
//     session's previous step, Section 3): its last block equals this chain's block at its length.
//     Its chain end is where this request's hit on the instance that took the parent most likely
//     ends.
//   * anc: the parent's parent and its parent, for the greedy's probe placement.
//   * base: the topmost request reached through par links.  This request's chain starts with the
//     base's whole chain, so on any cache its hit equals the base's hit unless the base is cached
//     in full; the probe derives such rows from the base's row.
// Every hit derived from these relations is exact as far as equal chained hashes mean equal
// prefixes, the same premise as the prefix search of the cached tables.
#include <algorithm>

#include "ps_internal.cuh"

namespace {

constexpr uint32_t kParentScan = 1024;  // chain positions scanned back from the end for a parent (16K tokens)

__device__ __forceinline__ uint32_t tab_home(uint64_t key, uint32_t n) {  // n is a power of two
  return (uint32_t)((key * 0x9E3779B97F4A7C15ull) >> 32) & (n - 1);
}

// Table of last-block hashes: each key keeps the earliest request whose chain ends with it.
__global__ void lastblock_build_kernel(psk::WindowDev w, psk::LastSlot* tab, uint32_t n) {
  for (uint32_t r = blockIdx.x * blockDim.x + threadIdx.x; r < w.R; r += gridDim.x * blockDim.x) {
    const uint64_t o = w.off[r], nb = w.off[r + 1] - o;
    if (nb == 0) continue;
    const unsigned long long key = w.hash[o + nb - 1];
    if (key == psk::kEmpty || key == psk::kTomb) continue;
    uint32_t b = tab_home(key, n);
    for (uint32_t p = 0; p < n; ++p) {
      const unsigned long long old = atomicCAS(&tab[b].key, (unsigned long long)psk::kEmpty, key);
      if (old == psk::kEmpty || old == key) {
        atomicMax(&tab[b].neg_idx, 0xFFFFFFFFu - r);
        break;
      }
      b = (b + 1) & (n - 1);
    }
  }
}

// Earliest request whose chain ends with key, -1 if none.  The first slot is loaded by the caller
// (first), so several lookups can be in flight together; collisions continue the linear probe.
__device__ __forceinline__ int32_t tab_resolve(const psk::LastSlot* tab, uint32_t n, uint64_t key, ulonglong2 first) {
  if (key == psk::kEmpty || key == psk::kTomb) return -1;
  uint32_t b = tab_home(key, n);
  ulonglong2 v = first;
  for (uint32_t p = 0; p < n; ++p) {
    if (v.x == key) return (int32_t)(0xFFFFFFFFu - (uint32_t)v.y);
    if (v.x == psk::kEmpty) return -1;
    b = (b + 1) & (n - 1);
    v = __ldg(reinterpret_cast<const ulonglong2*>(tab + b));
  }
  return -1;
}

constexpr int kScanPerLane = 8;  // parent-scan positions per lane and step (256 per warp step)
constexpr int kLcpGroup = 4;     // common-prefix searches advanced together
static_assert(psk::kLcpBack % kLcpGroup == 0, "whole groups of searches");

// One warp per request.  Chained block hashes (Section 7's prefix tree) make "block k equal" stand
// for "blocks 0..k equal", as in every prefix search of this library: the common prefix with an
// earlier request is a 32-ary first-miss search, and an earlier request whose last block equals
// this chain's block at its own length is a prefix of this chain.
//   lcp: the kLcpBack searches advance kLcpGroup at a time, one 32-ary step of each per round.
//   par: the last kParentScan positions are scanned back from the chain's end, 256 per warp step;
//        the deepest position whose block ends an earlier request of exactly that length gives the
//        parent.  A request whose parent lies further back is searched from scratch (exact).
__global__ void __launch_bounds__(256, 3)
relations_kernel(psk::WindowDev w, psk::DevModel m, const psk::LastSlot* tab, uint32_t n, psk::RowPre* rows) {
  const int lane = threadIdx.x & 31;
  const uint32_t wpb = blockDim.x >> 5;
  for (uint32_t r = blockIdx.x * wpb + (threadIdx.x >> 5); r < w.R; r += gridDim.x * wpb) {
    const uint64_t o = w.off[r];
    const uint64_t nb = w.off[r + 1] - o;
    const uint64_t* a = w.hash + o;
    uint32_t lcp[psk::kLcpBack];
#pragma unroll
    for (int g = 0; g < psk::kLcpBack; g += kLcpGroup) {
      // search of request r - 1 - d in [lo, hi]: positions below lo equal, hi differs (or is the end)
      uint32_t lo[kLcpGroup], hi[kLcpGroup];
      const uint64_t* bq[kLcpGroup];
#pragma unroll
      for (int u = 0; u < kLcpGroup; ++u) {
        const uint32_t d = (uint32_t)(g + u);
        lo[u] = hi[u] = 0u;
        bq[u] = a;
        if (r >= d + 1u) {
          const uint64_t oq = w.off[r - 1 - d];
          const uint64_t nq = w.off[r - d] - oq;
          bq[u] = w.hash + oq;
          hi[u] = (uint32_t)(nb < nq ? nb : nq);
        }
      }
      for (;;) {
        bool busy = false;
        bool ld[kLcpGroup];
        uint64_t va[kLcpGroup], vb[kLcpGroup];
#pragma unroll
        for (int u = 0; u < kLcpGroup; ++u) {
          const uint32_t span = hi[u] - lo[u];
          busy |= span != 0u;
          const uint32_t k = span <= 32u ? lo[u] + (uint32_t)lane
                                         : lo[u] + (uint32_t)(((uint64_t)(lane + 1) * span) >> 5) - 1u;
          ld[u] = span != 0u && k < hi[u];
          va[u] = ld[u] ? a[k] : 0ull;
          vb[u] = ld[u] ? bq[u][k] : 0ull;
        }
        if (!busy) break;  // warp-uniform
#pragma unroll
        for (int u = 0; u < kLcpGroup; ++u) {
          const uint32_t span = hi[u] - lo[u];
          if (span == 0u) continue;
          const unsigned miss = __ballot_sync(0xffffffffu, ld[u] && va[u] != vb[u]);
          if (span <= 32u) {
            lo[u] = hi[u] = miss ? lo[u] + (uint32_t)(__ffs(miss) - 1) : hi[u];
          } else if (!miss) {
            lo[u] = hi[u];
          } else {
            const uint64_t j = (uint64_t)(__ffs(miss) - 1);
            const uint32_t pj = lo[u] + (uint32_t)(((j + 1) * span) >> 5) - 1u;
            lo[u] = lo[u] + (uint32_t)((j * span) >> 5);
            hi[u] = pj;
          }
        }
      }
#pragma unroll
      for (int u = 0; u < kLcpGroup; ++u) lcp[g + u] = lo[u];
    }
    int32_t par = -1;
    uint32_t par_nb = 0;
    const uint64_t stop = nb > kParentScan ? nb - kParentScan : 0;
    for (uint64_t top = nb; top > stop && par < 0;) {
      const uint64_t lo_s = top - stop > 32u * kScanPerLane ? top - 32u * kScanPerLane : stop;
      uint64_t key[kScanPerLane];
      ulonglong2 first[kScanPerLane];
#pragma unroll
      for (int u = 0; u < kScanPerLane; ++u) {  // position top - 1 - lane - 32 u
        const uint64_t back = (uint64_t)lane + 32u * u;
        key[u] = back < top - lo_s ? a[top - 1 - back] : psk::kEmpty;
      }
#pragma unroll
      for (int u = 0; u < kScanPerLane; ++u)
        first[u] = (key[u] == psk::kEmpty || key[u] == psk::kTomb)
                       ? make_ulonglong2(psk::kEmpty, 0ull)
                       : __ldg(reinterpret_cast<const ulonglong2*>(tab + tab_home(key[u], n)));
#pragma unroll
      for (int u = 0; u < kScanPerLane; ++u) {
        const uint64_t back = (uint64_t)lane + 32u * u;
        const uint64_t k = top - 1 - back;
        int32_t cand = -1;
        if (back < top - lo_s) {
          const int32_t q = tab_resolve(tab, n, key[u], first[u]);
          if (q >= 0 && (uint32_t)q < r && w.off[q + 1] - w.off[q] == k + 1) cand = q;
        }
        const unsigned ok = __ballot_sync(0xffffffffu, cand >= 0);
        if (ok) {  // lower lanes hold deeper positions
          const int src = __ffs(ok) - 1;
          par = __shfl_sync(0xffffffffu, cand, src);
          par_nb = (uint32_t)(top - 32u * u - (uint64_t)src);
          break;
        }
      }
      top = lo_s;
    }
    if (lane == 0) {
      const psk::RowConst rc = psk::row_const(m, w.L[r], w.ttft_t[r], w.tpot_t[r]);
      psk::RowPre x{};
      x.off = o;
      x.nb = (uint32_t)nb;
      x.L = rc.L;
      x.t_cached = rc.t_cached;
      x.Z = rc.Z;
      x.etaZ = rc.etaZ;
      x.ttft_budget = rc.ttft_budget;
      x.tpot_target = rc.tpot_target;
#pragma unroll
      for (int d = 0; d < psk::kLcpBack; ++d) x.lcp[d] = lcp[d];
      x.par = par;
      x.par_nb = par_nb;
      x.base = -1;
      rows[r] = x;
    }
  }
}

// base and the two next ancestors of each request: follow the parent links (parents come
// earlier, so the walk ends).  Requests without a parent go to the list of rows the probe
// searches from scratch.
__global__ void base_kernel(uint32_t R, psk::RowPre* rows, psk::RowList list) {
  for (uint32_t r = blockIdx.x * blockDim.x + threadIdx.x; r < R; r += gridDim.x * blockDim.x) {
    int32_t a = rows[r].par;
    if (a < 0) list.rows[atomicAdd(list.count, 1u)] = r;  // searched from scratch
    int32_t anc[2] = {-1, -1};
    uint32_t anc_nb[2] = {0u, 0u};
    if (a >= 0) {
      anc[0] = rows[a].par;
      if (anc[0] >= 0) {
        anc_nb[0] = rows[a].par_nb;
        anc[1] = rows[anc[0]].par;
        if (anc[1] >= 0) anc_nb[1] = rows[anc[0]].par_nb;
      }
      for (int32_t p = rows[a].par; p >= 0; p = rows[a].par) a = p;
    }
    rows[r].base = a;
    rows[r].anc[0] = anc[0];
    rows[r].anc[1] = anc[1];
    rows[r].anc_nb[0] = anc_nb[0];
    rows[r].anc_nb[1] = anc_nb[1];
  }
}

}  // namespace

namespace pskl {

cudaError_t launch_relations(const psk::WindowDev& w, const psk::DevModel& m, psk::LastSlot* tab, uint32_t tab_n,
                             psk::RowPre* rows, psk::RowList list, int num_sms, cudaStream_t s) {
  cudaError_t e = cudaMemsetAsync(list.count, 0, sizeof(uint32_t), s);
  if (e != cudaSuccess || w.R == 0) return e;
  e = cudaMemsetAsync(tab, 0, (size_t)tab_n * sizeof(psk::LastSlot), s);
  if (e != cudaSuccess) return e;
  const int g1 = (int)std::min<uint64_t>((w.R + 255) / 256, (uint64_t)num_sms * 8);
  lastblock_build_kernel<<<g1, 256, 0, s>>>(w, tab, tab_n);
  e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  const int g2 = (int)((w.R + 7) / 8);  // one request per warp: blocks queue, so long rows balance out
  relations_kernel<<<g2, 256, 0, s>>>(w, m, tab, tab_n, rows);
  e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  base_kernel<<<g1, 256, 0, s>>>(w.R, rows, list);
  return cudaGetLastError();
}

}  // namespace pskl
