// Greedy in-window assignment (Algorithm 1 applied to the window's requests in arrival order).
//
// The paper's gateway decides each request online and updates the instance records along the
// request path before the next decision (Section 4, Metadata service; Section 7).  This kernel
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
              psk::StateSoA pending, psk::DevModel m, psk::DeltaSlot* delta, uint64_t delta_nslots,
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
        if (s_touched[i] && hc[k] < nb && psk::delta_contains(delta, delta_nslots, i, cn[k])) {
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
          return psk::delta_contains(delta, delta_nslots, i, key) ||
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
        if (!psk::delta_insert(delta, delta_nslots, j, w.hash[o + k])) atomicOr(err, psk::kErrDeltaFull);
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
                          uint64_t delta_nslots, int32_t* assign, uint8_t* path, uint32_t* hit_chosen,
                          uint32_t* err, uint32_t nt, cudaStream_t s) {
  const size_t smem = greedy_smem(I);
  cudaError_t e = cudaFuncSetAttribute(greedy_kernel<IPT, SEARCH>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       (int)smem);
  if (e != cudaSuccess) return e;
  greedy_kernel<IPT, SEARCH><<<1, nt, smem, s>>>(slots, ovf, tdesc, I, w, hit0, committed, pending, m, delta,
                                                 delta_nslots, assign, path, hit_chosen, err);
  return cudaGetLastError();
}


// ----------------------------------------------------------------------------------------------
// Prefix-closed caches (the probe's search mode): a software-pipelined greedy pass.
//
// On a prefix-closed cache the hit of a request is the first chain position not cached, and the
// union of prefix-closed sets has as first miss the largest of the sets' first misses.  The
// cached set of instance i while request s is decided is main_i plus the chains of the window's
// earlier requests assigned to i, so
//     hit(s, i) = max( first miss of main_i + delta_i(<= s - kLag),
//                      lcp(s, s - d) for each d = 1..kLag-1 such that request s - d went to i )
// where delta_i(<= s - kLag) holds the blocks inserted for requests up to s - kLag and lcp(s, s - d) is
// the common chain prefix (from the relations pass).  The first term is probed ahead of time, while
// earlier requests are still being decided, so no table access is on the per-request critical
// path.  The probe position is hit0, raised to the end of the request's parent (the deepest earlier
// request whose chain is a prefix of this one) on the instance that took the parent; a probe that
// finds the block cached hands the instance to a warp search.  Probes may also see inserts of
// requests s - kLag + 1 .. s - 1 (they land while the probe runs, in any order): any snapshot
// between delta(<= s - kLag) and delta(<= s - 1) gives a first miss between the two, and the max
// with the lcp terms is then exact all the same.
//
// Block 0 decides.  Per step r it evaluates row r (two block reductions: W_min, then the argmin)
// and besides:  loads hit0 of row r + 3;  places row r + 2's probe and loads the chain block there
// (instances with window inserts only);  issues row r + 1's probe (consumed after the first
// barrier);  publishes request r's pick as an insert job.  Blocks 1..kHelpers take the jobs
// round-robin (up to kHelpers jobs in flight), insert each job's chain blocks chain[h, nb) into
// delta_j and release the job's done flag; block 0 waits (bounded) for job r - (kLag - 2) before its
// row r + 2 probes go out; a dedicated signalling thread (the block's last warp
// owns no instances) publishes the jobs and does that wait, so the release and acquire orderings
// never hold up a thread with loads in flight.  Instance state lives in shared memory and is
// written only by the thread that owns the instance.

constexpr uint32_t kHelpers = 8;              // insert blocks beside the deciding block
constexpr uint32_t kRingAhead = 6;            // row constants are copied into the ring this many rows ahead
constexpr uint64_t kWaitNs = 1000000000ull;   // bound on any cross-block wait
constexpr unsigned long long kAbortJob = ~0ull;

struct PickKey {  // lexicographic (class, value, instance) element carrying the pair's hit
  uint32_t ci;
  uint32_t h;
  uint64_t v;
};

__device__ __forceinline__ bool pick_less(const PickKey& a, const PickKey& z) {
  return psk::key_less(psk::ArgKey{a.ci, a.v}, psk::ArgKey{z.ci, z.v});
}

__device__ __forceinline__ PickKey warp_pick(PickKey k) {
#pragma unroll
  for (int s = 16; s > 0; s >>= 1) {
    PickKey o;
    o.ci = __shfl_xor_sync(0xffffffffu, k.ci, s);
    o.h = __shfl_xor_sync(0xffffffffu, k.h, s);
    o.v = __shfl_xor_sync(0xffffffffu, k.v, s);
    if (pick_less(o, k)) k = o;
  }
  return k;
}

__device__ __forceinline__ psk::RowConst row_of(const psk::RowPre& x) {
  psk::RowConst rc;
  rc.t_cached = x.t_cached;
  rc.Z = x.Z;
  rc.etaZ = x.etaZ;
  rc.ttft_budget = x.ttft_budget;
  rc.tpot_target = x.tpot_target;
  rc.L = x.L;
  return rc;
}

// Blocks 1..kHelpers: block b inserts the chain tails of jobs b - 1, b - 1 + kHelpers, ... and
// releases each job's done flag once all its blocks are in.
__device__ void insert_helper(const psk::RowPre* __restrict__ rows, const uint64_t* __restrict__ hash, uint32_t R,
                              psk::DeltaSlot* delta, uint64_t nslots, uint32_t* err, const psk::GreedySync& sync) {
  __shared__ unsigned long long s_job;
  const uint32_t t = threadIdx.x;
  for (uint32_t job = blockIdx.x - 1; job < R; job += kHelpers) {
    if (t == 0) {
      const uint64_t t0 = psk::globaltimer_ns();
      unsigned long long jb = kAbortJob;
      for (;;) {
        if (psk::ld_acquire_u32(sync.pub) > job) {
          jb = __ldcg(sync.jobs + job);
          break;
        }
        if (psk::globaltimer_ns() - t0 > kWaitNs) {
          atomicOr(err, psk::kErrTimeout);
          break;
        }
        __nanosleep(32);
      }
      s_job = jb;
    }
    __syncthreads();
    const unsigned long long jb = s_job;
    if (jb == kAbortJob) return;  // block-uniform
    const uint32_t j = (uint32_t)jb;
    const uint32_t hj = (uint32_t)(jb >> 32);
    // rows >= job + kLag are the only ones that read this job's inserts
    if (j != 0xFFFFFFFFu && job + psk::kLag < R) {
      const uint64_t off = __ldg(&rows[job].off);
      const uint32_t nb = __ldg(&rows[job].nb);
      for (uint64_t p = hj + t; p < nb; p += blockDim.x)
        if (!psk::delta_insert(delta, nslots, j, __ldg(hash + off + p))) atomicOr(err, psk::kErrDeltaFull);
    }
    __syncthreads();
    if (t == 0) {
      __threadfence();  // every thread's inserts before the flag
      psk::st_release_u32(sync.done + job, 1u);
    }
  }
}

template <int IPT>
__global__ void __launch_bounds__(544, 1)
greedy_search_kernel(const psk::RowPre* __restrict__ rows, const uint64_t* __restrict__ hash, uint32_t R, uint32_t I,
                     const uint32_t* __restrict__ hit0, const float* __restrict__ tpf0, psk::StateSoA committed, psk::StateSoA pending,
                     psk::DevModel m, psk::DeltaSlot* delta, uint64_t nslots, int32_t* assign,
                     uint8_t* __restrict__ path, uint32_t* __restrict__ hit_chosen, uint32_t* err,
                     psk::GreedySync sync) {
  if (blockIdx.x > 0) {
    insert_helper(rows, hash, R, delta, nslots, err, sync);
    return;
  }
  extern __shared__ unsigned long long smem_raw[];
  int64_t* s_q = reinterpret_cast<int64_t*>(smem_raw);
  int64_t* s_S = s_q + I;
  int64_t* s_M = s_S + I;
  int32_t* s_b = reinterpret_cast<int32_t*>(s_M + I);
  int32_t* s_qr = s_b + I;
  int32_t* s_Bmax = s_qr + I;
  uint32_t* s_end = reinterpret_cast<uint32_t*>(s_Bmax + I);  // chain end of the last request on i
  uint32_t* s_wres = s_end + I;                                // search start / result per instance
  uint32_t* s_walk = s_wres + I;                               // instances handed to a warp search
  psk::InstTerms* s_it = reinterpret_cast<psk::InstTerms*>(s_walk + I);
  uint8_t* s_touched = reinterpret_cast<uint8_t*>(s_it + I);
  __shared__ psk::RowPre s_row[8];  // rows r .. r + kRingAhead (a ring of 8 so no reader is overtaken)
  __shared__ float s_red_w[32];
  __shared__ int s_red_a[32];
  __shared__ PickKey s_red_k[32];
  __shared__ uint32_t s_nwalk[2];

  const int t = threadIdx.x;
  const int NT = blockDim.x;
  const int NTI = NT - 32;  // threads owning instances; the last warp signals
  const bool sig = t == NTI;
  const int lane = t & 31;
  const int warp = t >> 5;
  const int NW = NT >> 5;
  // instance k of this thread (out of range for the signalling warp)
  auto own = [&](int k) -> uint32_t { return t < NTI ? (uint32_t)(t + k * NTI) : 0xFFFFFFFFu; };

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
  if (t < kRingAhead * psk::kRowWords) {  // rows 0 .. kRingAhead - 1
    const uint32_t rr = (uint32_t)(t / psk::kRowWords);
    if (rr < R)
      reinterpret_cast<uint4*>(&s_row[rr])[t % psk::kRowWords] =
          __ldg(reinterpret_cast<const uint4*>(rows + rr) + (t % psk::kRowWords));
  }
  if (t < 2) s_nwalk[t] = 0;

  // hit and T_pf at that hit of rows r .. r + 2 (T_pf from the probe; kNoTpfBits once the greedy
  // changed the hit)
  uint32_t hr[IPT], h1[IPT], h2[IPT];
  float tr[IPT], t1[IPT], t2[IPT];
  uint64_t key1[IPT];
  bool need1[IPT];
#pragma unroll
  for (int k = 0; k < IPT; ++k) {
    const uint32_t i = own(k);
    hr[k] = (i < I && R > 0) ? __ldg(hit0 + i) : 0u;
    h1[k] = (i < I && R > 1) ? __ldg(hit0 + (uint64_t)I + i) : 0u;
    h2[k] = (i < I && R > 2) ? __ldg(hit0 + 2ull * I + i) : 0u;
    tr[k] = (i < I && R > 0) ? __ldg(tpf0 + i) : 0.0f;
    t1[k] = (i < I && R > 1) ? __ldg(tpf0 + (uint64_t)I + i) : 0.0f;
    t2[k] = (i < I && R > 2) ? __ldg(tpf0 + 2ull * I + i) : 0.0f;
    key1[k] = 0;
    need1[k] = false;
  }
  int32_t jm[psk::kLcpBack];  // jm[d] = pick of request r - 1 - d
#pragma unroll
  for (int d = 0; d < psk::kLcpBack; ++d) jm[d] = -1;
  int32_t jp_pre[3] = {-1, -1, -1};  // picks of row r + 2's parent and two next ancestors, loaded a step ahead
  bool timed_out = false;
  __syncthreads();

  for (uint32_t r = 0; r < R; ++r) {
    const psk::RowPre& cur = s_row[r & 7];
    const uint32_t nb = cur.nb;
    // ---- P0: ring refill, stages A-C, corrections and row evaluation -----------------------------
    // Refill the ring kRingAhead rows ahead: one copy group per step (empty past the window's end),
    // waited for two steps later, so the copy's latency stays off the step.
    if (t < psk::kRowWords) {
      if (r + kRingAhead < R)
        psk::cp_async16(reinterpret_cast<uint4*>(&s_row[(r + kRingAhead) & 7]) + t,
                        reinterpret_cast<const uint4*>(rows + r + kRingAhead) + t);
      psk::cp_async_commit();
    }
    // The signalling thread starts reading job r - (kLag - 2)'s done flag now; it is checked before
    // the second barrier.
    uint32_t done_seen = 1u;
    if (sig && r >= psk::kLag - 2 && !timed_out) done_seen = psk::ld_acquire_u32(sync.done + (r - (psk::kLag - 2)));
    // picks of row r + 3's ancestors when they are old enough to be in global memory (instance
    // threads only: the signalling thread keeps no loads in flight)
    int32_t jp_next[3] = {-1, -1, -1};
    if (t < NTI && r + 3 < R) {
      const psk::RowPre& x3 = s_row[(r + 3) & 7];
      const int32_t a3[3] = {x3.par, x3.anc[0], x3.anc[1]};
#pragma unroll
      for (int q = 0; q < 3; ++q)
        if (a3[q] >= 0 && (int64_t)a3[q] <= (int64_t)r - (psk::kLag - 1)) jp_next[q] = __ldcg(assign + a3[q]);
    }
    uint32_t h3[IPT];
    float t3[IPT];
#pragma unroll
    for (int k = 0; k < IPT; ++k) {
      const uint32_t i = own(k);
      h3[k] = (i < I && r + 3 < R) ? __ldg(hit0 + (uint64_t)(r + 3) * I + i) : 0u;
      t3[k] = (i < I && r + 3 < R) ? __ldg(tpf0 + (uint64_t)(r + 3) * I + i) : 0.0f;
    }
    uint64_t key2[IPT];
    bool need2[IPT];
    if (r + 2 < R) {
      const psk::RowPre& x2 = s_row[(r + 2) & 7];
      // An ancestor's chain is a prefix of this one; on the instance that took it, the probe goes
      // to its end.  It counts only if its inserts are in every probe snapshot: a <= (r + 2) - kLag,
      // i.e. its distance d = r + 2 - a is at least kLag; its pick is jm[d - 3] while that is still
      // in registers, else the one loaded from global memory a step ahead.
      const int32_t a2[3] = {x2.par, x2.anc[0], x2.anc[1]};
      const uint32_t a2nb[3] = {x2.par_nb, x2.anc_nb[0], x2.anc_nb[1]};
      int32_t jp[3];
#pragma unroll
      for (int q = 0; q < 3; ++q) {
        const int64_t a = a2[q];
        jp[q] = -1;
        if (a >= 0) {
          const int64_t d = (int64_t)r + 2 - a;
          if (d == psk::kLag) jp[q] = jm[psk::kLag - 3];
          else if (d == psk::kLag + 1) jp[q] = jm[psk::kLag - 2];
          else if (d >= psk::kLag + 2) jp[q] = jp_pre[q];
        }
      }
#pragma unroll
      for (int k = 0; k < IPT; ++k) {
        const uint32_t i = own(k);
        uint32_t pos = h2[k];
#pragma unroll
        for (int q = 0; q < 3; ++q)
          if ((int32_t)i == jp[q] && a2nb[q] > pos) pos = a2nb[q];
        need2[k] = i < I && s_touched[i] && pos < x2.nb;
        key2[k] = need2[k] ? __ldg(hash + x2.off + pos) : 0ull;
        if (pos != h2[k]) t2[k] = __uint_as_float(psk::kNoTpfBits);
        h2[k] = pos;
      }
    } else {
#pragma unroll
      for (int k = 0; k < IPT; ++k) {
        need2[k] = false;
        key2[k] = 0;
      }
    }
    ulonglong2 pv0[IPT], pv1[IPT];
    uint64_t home1[IPT];
#pragma unroll
    for (int k = 0; k < IPT; ++k) {
      const uint32_t i = own(k);
      if (need1[k]) {
        home1[k] = psk::delta_home(key1[k], nslots);
        pv0[k] = __ldcg(reinterpret_cast<const ulonglong2*>(delta + home1[k]));
        pv1[k] = __ldcg(reinterpret_cast<const ulonglong2*>(delta + psk::delta_next(home1[k], nslots)));
      } else {
        home1[k] = 0;
        pv0[k] = make_ulonglong2(0ull, 0ull);
        pv1[k] = make_ulonglong2(0ull, 0ull);
      }
    }

    // Pass 1: hit corrections, W and the capacity guard; W_min over A.
    const psk::RowConst rc = row_of(cur);
    psk::PairW ev[IPT];
    float wmin = INFINITY;
    bool anyA = false;
#pragma unroll
    for (int k = 0; k < IPT; ++k) {
      const uint32_t i = own(k);
      if (i < I) {
        uint32_t h = hr[k];
#pragma unroll
        for (int d = 0; d < psk::kLcpBack; ++d)
          if ((int32_t)i == jm[d] && cur.lcp[d] > h) h = cur.lcp[d];
        const float tp = h == hr[k] ? tr[k] : __uint_as_float(psk::kNoTpfBits);
        hr[k] = h;
        ev[k] = psk::pair_w(m, rc, h, tp, s_it[i], s_S[i], s_M[i]);
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

    // ---- P1: W_min, admission classes, argmin; row r + 1's probes; wait for job r - 3 -------------
    {
      const float v = lane < NW ? s_red_w[lane] : INFINITY;
      const bool a = lane < NW ? (s_red_a[lane] != 0) : false;
      wmin = psk::warp_fmin(v);
      anyA = __any_sync(0xffffffffu, a);
    }
    // Pass 2: latencies and the admission class of the pairs in C only; the argmin key.
    PickKey best{psk::kNoKeyCi, 0u, ~0ull};
#pragma unroll
    for (int k = 0; k < IPT; ++k) {
      const uint32_t i = own(k);
      if (i < I && ev[k].inA && psk::pair_in_c(rc, ev[k].W, wmin)) {
        const int64_t q = s_q[i];
        float tpot, ttft;
        psk::pair_lat(m, rc, ev[k], s_it[i], q, s_S[i], &tpot, &ttft);
        const uint32_t cls = psk::pair_admitted(m, rc, tpot, ttft) ? 0u : 1u;
        const PickKey kk{(cls << 28) | i, hr[k], psk::pair_value(cls, hr[k], s_b[i], s_qr[i], q, ev[k].n)};
        if (pick_less(kk, best)) best = kk;
      }
    }
    best = warp_pick(best);
    if (lane == 0) s_red_k[warp] = best;
    bool walked[IPT];
#pragma unroll
    for (int k = 0; k < IPT; ++k) {
      const uint32_t i = own(k);
      walked[k] = false;
      if (need1[k]) {
        int v = psk::delta_slot_verdict(pv0[k], key1[k], i + 1);
        if (v < 0) v = psk::delta_slot_verdict(pv1[k], key1[k], i + 1);
        const bool present = v >= 0 ? v == 1
                                    : psk::delta_contains_from(delta, nslots, i, key1[k],
                                                               psk::delta_next(psk::delta_next(home1[k], nslots), nslots));
        if (present) {
          const uint32_t x = atomicAdd(&s_nwalk[(r + 1) & 1], 1u);
          s_walk[x] = i;
          s_wres[i] = h1[k];
          walked[k] = true;
        }
      }
    }
    // rows <= r + kRingAhead - 2 are in (the next step reads row r + 4)
    if (t < psk::kRowWords) psk::cp_async_wait_group<2>();
    // Row r + 2's probes (issued in the next step) need every insert of requests <= r + 2 - kLag;
    // the earlier jobs were waited for in earlier steps.
    if (sig && done_seen == 0u) {
      const uint64_t t0 = psk::globaltimer_ns();
      while (psk::ld_acquire_u32(sync.done + (r - (psk::kLag - 2))) == 0u) {
        if (psk::globaltimer_ns() - t0 > kWaitNs) {
          atomicOr(err, psk::kErrTimeout);
          timed_out = true;
          break;
        }
      }
    }
    __syncthreads();  // (D)

    // ---- P2: the pick, its state, its insert job; searches for row r + 1 --------------------------
    {
      const PickKey o = lane < NW ? s_red_k[lane] : PickKey{psk::kNoKeyCi, 0u, ~0ull};
      best = warp_pick(o);
    }
    const bool pick = anyA && best.ci != psk::kNoKeyCi;
    const uint32_t j = best.ci & 0x0FFFFFFFu;
    const uint32_t hj = pick ? best.h : 0u;
    if (sig) {
      assign[r] = pick ? (int32_t)j : -1;
      path[r] = pick ? (uint8_t)(best.ci >> 28) : (uint8_t)2;
      hit_chosen[r] = hj;
      s_nwalk[r & 1] = 0;
      sync.jobs[r] = ((unsigned long long)hj << 32) | (pick ? j : 0xFFFFFFFFu);
      psk::st_release_u32(sync.pub, r + 1);
    }
    if (pick && (j % (uint32_t)NTI) == (uint32_t)t) {
      s_qr[j] += 1;
      s_q[j] += (int64_t)rc.L - 16 * (int64_t)hj;
      s_S[j] += (int64_t)rc.L;
      s_end[j] = nb;
      s_touched[j] = 1;
      s_it[j] = psk::inst_terms(m, s_b[j], s_qr[j], s_q[j], s_Bmax[j]);
    }
    const uint32_t nwalk = r + 1 < R ? s_nwalk[(r + 1) & 1] : 0u;
    if (nwalk) {
      const psk::RowPre& x1 = s_row[(r + 1) & 7];
      const uint64_t xoff = x1.off, xnb = x1.nb;
      for (uint32_t x = warp; x < nwalk; x += NW) {
        const uint32_t i = s_walk[x];
        auto cached = [&](uint64_t k) {
          return k < xnb && psk::delta_contains(delta, nslots, i, __ldg(hash + xoff + k));
        };
        const uint64_t hnew = psk::warp_first_miss_search_hint((uint64_t)s_wres[i] + 1, xnb, s_end[i], cached);
        __syncwarp();
        if (lane == 0) s_wres[i] = (uint32_t)hnew;
      }
      __syncthreads();  // (E) search results visible to the owners
#pragma unroll
      for (int k = 0; k < IPT; ++k)
        if (walked[k]) {
          h1[k] = s_wres[own(k)];
          t1[k] = __uint_as_float(psk::kNoTpfBits);
        }
    }
#pragma unroll
    for (int k = 0; k < IPT; ++k) {
      tr[k] = t1[k];
      t1[k] = t2[k];
      t2[k] = t3[k];
      hr[k] = h1[k];
      h1[k] = h2[k];
      key1[k] = key2[k];
      need1[k] = need2[k];
      h2[k] = h3[k];
    }
#pragma unroll
    for (int d = psk::kLcpBack - 1; d > 0; --d) jm[d] = jm[d - 1];
    jm[0] = pick ? (int32_t)j : -1;
#pragma unroll
    for (int q = 0; q < 3; ++q) jp_pre[q] = jp_next[q];
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

size_t greedy_search_smem(uint32_t I) {
  return (size_t)I * (3 * sizeof(int64_t) + 3 * sizeof(int32_t) + 3 * sizeof(uint32_t) + sizeof(psk::InstTerms) + 1) + 16;
}

template <int IPT>
cudaError_t greedy_search_launch(const psk::RowPre* rows, const psk::WindowDev& w, uint32_t I, const uint32_t* hit0,
                                 const float* tpf0, psk::StateSoA committed, psk::StateSoA pending, const psk::DevModel& m,
                                 psk::DeltaSlot* delta, uint64_t nslots, int32_t* assign, uint8_t* path,
                                 uint32_t* hit_chosen, uint32_t* err, const psk::GreedySync& sync, uint32_t nt,
                                 cudaStream_t s) {
  const size_t smem = greedy_search_smem(I);
  cudaError_t e = cudaFuncSetAttribute(greedy_search_kernel<IPT>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (e != cudaSuccess) return e;
  const uint64_t* hash = w.hash;
  uint32_t R = w.R;
  psk::StateSoA c = committed, p = pending;
  psk::DevModel mm = m;
  psk::GreedySync sy = sync;
  void* args[] = {(void*)&rows, (void*)&hash, (void*)&R, (void*)&I, (void*)&hit0, (void*)&tpf0, (void*)&c, (void*)&p,
                  (void*)&mm, (void*)&delta, (void*)&nslots, (void*)&assign, (void*)&path, (void*)&hit_chosen,
                  (void*)&err, (void*)&sy};
  // all 1 + kHelpers blocks must be resident at once: they wait on one another
  return cudaLaunchCooperativeKernel((const void*)greedy_search_kernel<IPT>, dim3(1 + kHelpers), dim3(nt), args, smem, s);
}

}  // namespace

namespace pskl {

cudaError_t launch_greedy(const uint64_t* slots, const uint64_t* ovf, const psk::TableDesc* tdesc, uint32_t I,
                          const psk::WindowDev& w, const uint32_t* hit0, psk::StateSoA committed,
                          psk::StateSoA pending, const psk::DevModel& m, psk::DeltaSlot* delta,
                          uint64_t delta_nslots, int32_t* assign, uint8_t* path, uint32_t* hit_chosen,
                          uint32_t* err, int search, cudaStream_t s) {
  uint32_t nt = (I + 31) / 32 * 32;
  if (nt > 1024) nt = 1024;
  const uint32_t ipt = (I + nt - 1) / nt;
#define PS_GREEDY(IPT)                                                                                         \
  return search ? greedy_launch<IPT, true>(slots, ovf, tdesc, I, w, hit0, committed, pending, m, delta,        \
                                           delta_nslots, assign, path, hit_chosen, err, nt, s)                   \
                : greedy_launch<IPT, false>(slots, ovf, tdesc, I, w, hit0, committed, pending, m, delta,       \
                                            delta_nslots, assign, path, hit_chosen, err, nt, s)
  if (ipt <= 1) PS_GREEDY(1);
  if (ipt <= 2) PS_GREEDY(2);
  if (ipt <= 4) PS_GREEDY(4);
#undef PS_GREEDY
  return cudaErrorInvalidValue;
}

cudaError_t launch_greedy_search(const psk::RowPre* rows, const psk::WindowDev& w, uint32_t I, const uint32_t* hit0,
                                 const float* tpf0, psk::StateSoA committed, psk::StateSoA pending, const psk::DevModel& m,
                                 psk::DeltaSlot* delta, uint64_t delta_nslots, int32_t* assign, uint8_t* path,
                                 uint32_t* hit_chosen, uint32_t* err, const psk::GreedySync& sync, cudaStream_t s) {
  cudaError_t e = w.R ? cudaMemsetAsync(sync.done, 0, (size_t)w.R * sizeof(uint32_t), s) : cudaSuccess;
  if (e == cudaSuccess) e = cudaMemsetAsync(sync.pub, 0, sizeof(uint32_t), s);
  if (e != cudaSuccess) return e;
  // up to 512 threads each owning IPT instances (IPT = 1, 2 or 4 for I up to 2048), plus one
  // signalling warp
  const uint32_t ipt = I <= 512 ? 1u : (I <= 1024 ? 2u : 4u);
  const uint32_t nt = ((I + ipt - 1) / ipt + 31) / 32 * 32 + 32;
#define PS_GREEDY_S(IPT)                                                                                        \
  return greedy_search_launch<IPT>(rows, w, I, hit0, tpf0, committed, pending, m, delta, delta_nslots, assign, path,  \
                                   hit_chosen, err, sync, nt, s)
  if (ipt == 1) PS_GREEDY_S(1);
  if (ipt == 2) PS_GREEDY_S(2);
  if (ipt == 4 && I <= 2048) PS_GREEDY_S(4);
#undef PS_GREEDY_S
  return cudaErrorInvalidValue;
}

// The delta table only holds one window's blocks: clear it whole after each window.
cudaError_t launch_delta_clear(psk::DeltaSlot* delta, uint64_t nslots, cudaStream_t s) {
  return cudaMemsetAsync(delta, 0, nslots * sizeof(psk::DeltaSlot), s);
}

}  // namespace pskl
