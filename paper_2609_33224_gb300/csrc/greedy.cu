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

// Per-warp (key, tie) partials -> the block's minimum, reduced by every warp.
__device__ __forceinline__ void cross_warp_pick(const uint4* s_k, int nw, uint64_t* key, uint32_t* tie) {
  const int lane = threadIdx.x & 31;
  const uint4 pk = lane < nw ? s_k[lane] : make_uint4(0xFFFFFFFFu, 0xFFFFFFFFu, 0xFFFFFFFFu, 0u);
  uint32_t h;
  psk::warp_pick_min(((uint64_t)pk.y << 32) | pk.x, pk.z, pk.w, key, tie, &h);
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
  __shared__ uint4 s_red_k[32];
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
    // Pass 2: admission classes and the packed (class, value) key with its tie word.
    uint64_t bkey = psk::kNoKey;
    uint32_t btie = 0xFFFFFFFFu;
#pragma unroll
    for (int k = 0; k < IPT; ++k) {
      const uint32_t i = t + k * NT;
      if (i < I && ev[k].inA) {
        const uint32_t cls = psk::pair_class(m, rc, ev[k], wmin);
        if (cls <= 1u) {
          uint64_t key;
          uint32_t tie = i;
          if (cls == 0u) {
            key = psk::packed_key(0u, psk::value_in_t(m, psk::key0_bits(m, s_b[i], s_qr[i]), hc[k], ev[k].tpot,
                                                      rc.tpot_target));
            tie = psk::tie_in_t(m, i, s_qr[i]);
          } else {
            const int32_t Bp = s_b[i] + s_qr[i] + 1;
            key = psk::packed_key(1u, psk::value_fallback(m, (uint64_t)(s_q[i] + ev[k].n), (uint32_t)Bp,
                                                          psk::dcq_key0(s_b[i], s_qr[i]), hc[k]));
          }
          if (key < bkey || (key == bkey && tie < btie)) {
            bkey = key;
            btie = tie;
          }
        }
      }
    }
    {
      uint64_t wk;
      uint32_t wt, wh;
      psk::warp_pick_min(bkey, btie, 0u, &wk, &wt, &wh);
      if (lane == 0) s_red_k[warp] = make_uint4((uint32_t)wk, (uint32_t)(wk >> 32), wt, 0u);
    }
    __syncthreads();  // (D)
    uint64_t bk;
    uint32_t bt;
    cross_warp_pick(s_red_k, NW, &bk, &bt);
    const bool pick = anyA && bk != psk::kNoKey;
    const uint32_t j = bt & psk::kTieInstMask;
    const uint32_t hj = pick ? s_h[j] : 0u;
    if (t == 0) {
      assign[r] = pick ? (int32_t)j : -1;
      path[r] = pick ? (uint8_t)(bk >> 62) : (uint8_t)2;
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
// Prefix-closed caches (the probe's search mode): a pipelined greedy pass over three kinds of
// thread block in one cooperative launch.
//
// On a prefix-closed cache the hit of a request is the first chain position not cached, and the
// union of prefix-closed sets has as first miss the largest of the sets' first misses.  The
// cached set of instance i while request s is decided is main_i plus the chains of the window's
// earlier requests assigned to i, so
//     hit(s, i) = max( first miss of main_i + delta_i(<= s - kLag),
//                      lcp(s, s - d) for each d = 1..kLag-1 such that request s - d went to i )
// where delta_i(<= s - kLag) holds the blocks inserted for requests up to s - kLag and lcp(s, s - d) is
// the common chain prefix (from the relations pass).
//
//   Deciding block (block 0).  Per request r: reads row r's probed hits (first term above) from a
//   shared-memory ring that was filled by asynchronous copies two steps earlier, raises the hits of
//   the instances that took requests r - 1 .. r - kLag + 1 to the common prefix, evaluates the row
//   (capacity guard and W, block reduction to W_min; recompute filter, latencies, admission class
//   and key of the pairs in C, block reduction to the pick), updates the pick's state and publishes
//   the decision as an insert job.  No table access is on its per-request path.
//   Insert blocks.  Take the jobs round-robin (up to kInsertBlocks in flight), insert each job's
//   chain blocks chain[h, nb) into delta_j and release the job's done flag.
//   Probe blocks.  Take the rows round-robin.  For row s they wait until the jobs <= s - kLag are
//   done, replay those jobs (which instances have window inserts, where their last chain ended,
//   which instances took s's ancestors), then per instance start from hit0, raise the position to
//   the end of an ancestor's chain on the instance that took it (its chain is a prefix of s's, and
//   its inserts are in), probe the delta table there when the instance has window inserts, hand the
//   instances whose block is present to a warp search over the delta, and release the row's ready
//   flag.  The main table is never probed here: positions past hit0 are absent from a
//   prefix-closed main table.  Inserts of requests s - kLag + 1 .. s - 1 may land while a probe
//   runs, in any order: any snapshot between delta(<= s - kLag) and delta(<= s - 1) gives a first
//   miss between the two sets' first misses, and the max with the lcp terms is exact all the same.
// Every cross-block wait is bounded (GreedySync::wait_ns, 1 s unless the caller set another limit);
// on expiry the waiter records PS_ERR_TIMEOUT and stops waiting, so the launch always ends.  Instance state lives in the deciding block's shared
// memory and is written only by the thread that owns the instance.

constexpr uint32_t kInsertBlocks = 8;         // insert blocks
constexpr uint32_t kProbeBlocks = 16;         // probe blocks
constexpr uint32_t kRingAhead = 6;            // row constants are copied into the ring this many rows ahead
constexpr unsigned long long kJobValid = 1ull << 63;  // a published job word (0 = not yet published)

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

// Bounded spin until *flag != 0 (acquire).  false after limit_ns (and the error bit is set).
__device__ __forceinline__ bool wait_flag(const uint32_t* flag, uint32_t* err, uint64_t limit_ns) {
  if (psk::ld_acquire_u32(flag) != 0u) return true;
  const uint64_t t0 = psk::globaltimer_ns();
  while (psk::ld_acquire_u32(flag) == 0u) {
    if (psk::globaltimer_ns() - t0 > limit_ns) {
      atomicOr(err, psk::kErrTimeout);
      return false;
    }
    __nanosleep(32);
  }
  return true;
}

// Bounded wait for a published job word; 0 after limit_ns (and the error bit is set).
__device__ __forceinline__ unsigned long long wait_job(const unsigned long long* job, uint32_t* err,
                                                       uint64_t limit_ns) {
  unsigned long long v = psk::ld_relaxed_u64(job);
  if (v & kJobValid) return v;
  const uint64_t t0 = psk::globaltimer_ns();
  for (;;) {
    v = psk::ld_relaxed_u64(job);
    if (v & kJobValid) return v;
    if (psk::globaltimer_ns() - t0 > limit_ns) {
      atomicOr(err, psk::kErrTimeout);
      return 0ull;
    }
    __nanosleep(32);
  }
}

__device__ __forceinline__ uint32_t job_pick(unsigned long long jb) { return (uint32_t)jb; }
__device__ __forceinline__ uint32_t job_hit(unsigned long long jb) { return (uint32_t)(jb >> 32) & 0x7FFFFFFFu; }

// Insert blocks: block b inserts the chain tails of jobs b - 1, b - 1 + kInsertBlocks, ... and
// releases each job's done flag once all its blocks are in.
__device__ void insert_blocks(const psk::RowPre* __restrict__ rows, const uint64_t* __restrict__ hash, uint32_t R,
                              psk::DeltaSlot* delta, uint64_t nslots, uint32_t* err, const psk::GreedySync& sync) {
  __shared__ unsigned long long s_job;
  const uint32_t t = threadIdx.x;
  for (uint32_t job = blockIdx.x - 1; job < R; job += kInsertBlocks) {
    if (t == 0) s_job = wait_job(sync.jobs + job, err, sync.wait_ns);
    __syncthreads();
    const unsigned long long jb = s_job;
    if (jb == 0ull) return;  // block-uniform: timed out
    const uint32_t j = job_pick(jb);
    const uint32_t hj = job_hit(jb);
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

// Probe blocks: block p probes rows p, p + kProbeBlocks, ... in order (see the section comment).
// Per row, everything that does not need the window's inserts comes first: replaying the published
// jobs <= s - kLag (which instances have window inserts, their last chain end, the picks of the
// row's ancestors), the hit0 row, the probe positions and the chain blocks there.  Only then does the
// block wait until those jobs' inserts are done, so after the wait one delta lookup per instance
// (and, rarely, a warp search) is left before the row is released.
template <int IPT>
__device__ void probe_rows(const psk::RowPre* __restrict__ rows, const uint64_t* __restrict__ hash, uint32_t R,
                           uint32_t I, const uint32_t* __restrict__ hit0, const float* __restrict__ tpf0,
                           const psk::DeltaSlot* delta, uint64_t nslots, uint32_t* err, const psk::GreedySync& sync,
                           unsigned long long* smem_raw) {
  uint32_t* s_end = reinterpret_cast<uint32_t*>(smem_raw);  // chain end of the last job on i (0 = none)
  uint32_t* s_res = s_end + I;                               // search start / result per instance
  uint32_t* s_walk = s_res + I;                              // instances handed to a warp search
  __shared__ uint32_t s_nwalk;
  __shared__ int32_t s_ja[3];       // picks of the row's ancestors old enough to count (-1: none)
  __shared__ uint32_t s_jnb[3];     // their chain lengths
  __shared__ uint32_t s_replayed;   // jobs [0, s_replayed) are published and replayed
  __shared__ uint32_t s_done;       // jobs [0, s_done) have their inserts in the delta table
  __shared__ int s_abort;
  const uint32_t t = threadIdx.x;
  const uint32_t NT = blockDim.x;
  const int lane = t & 31, warp = t >> 5, NW = NT >> 5;
  for (uint32_t i = t; i < I; i += NT) s_end[i] = 0u;
  if (t == 0) {
    s_replayed = 0;
    s_done = 0;
    s_nwalk = 0;
    s_abort = 0;
  }
  __syncthreads();
  for (uint32_t s = blockIdx.x - 1 - kInsertBlocks; s < R; s += kProbeBlocks) {
    const uint64_t off = __ldg(&rows[s].off);
    const uint32_t nb = __ldg(&rows[s].nb);
    const int64_t need = (int64_t)s - psk::kLag + 1;  // jobs [0, need) count for this row
    if (warp == 0) {
      // Replay the published jobs [replayed, need), 32 at a time; for each instance the latest of
      // them sets its chain end.
      uint32_t f = s_replayed;
      bool abort = false;
      while ((int64_t)f < need && !abort) {
        const uint32_t x = f + (uint32_t)lane;
        const bool mine = (int64_t)x < need;
        unsigned long long jb = 0ull;
        if (mine) jb = wait_job(sync.jobs + x, err, sync.wait_ns);
        abort = __any_sync(0xffffffffu, mine && jb == 0ull);
        if (abort) break;
        const uint32_t j = mine ? job_pick(jb) : 0xFFFFFFFFu;
        const uint32_t nbx = mine ? __ldg(&rows[x].nb) : 0u;
        const unsigned same = __match_any_sync(0xffffffffu, j);
        if (mine && j < I && (31 - __clz(same)) == lane) s_end[j] = nbx;
        const uint32_t n = (int64_t)f + 32 <= need ? 32u : (uint32_t)(need - (int64_t)f);
        f += n;
      }
      if (lane == 0) {
        s_replayed = f;
        s_abort = abort ? 1 : 0;
        const int32_t a[3] = {__ldg(&rows[s].par), __ldg(&rows[s].anc[0]), __ldg(&rows[s].anc[1])};
        const uint32_t anb[3] = {__ldg(&rows[s].par_nb), __ldg(&rows[s].anc_nb[0]), __ldg(&rows[s].anc_nb[1])};
#pragma unroll
        for (int q = 0; q < 3; ++q) {
          s_ja[q] = -1;
          s_jnb[q] = anb[q];
          if (!abort && a[q] >= 0 && (int64_t)a[q] < need) {
            const uint32_t j = job_pick(psk::ld_relaxed_u64(sync.jobs + a[q]));
            if (j < I) s_ja[q] = (int32_t)j;
          }
        }
      }
    }
    __syncthreads();
    if (s_abort) return;  // block-uniform
    const int32_t ja0 = s_ja[0], ja1 = s_ja[1], ja2 = s_ja[2];
    const uint32_t jn0 = s_jnb[0], jn1 = s_jnb[1], jn2 = s_jnb[2];
    uint32_t h0[IPT], pos[IPT];
    float tp0[IPT];
    uint64_t key[IPT];
    bool probe[IPT], walk[IPT];
#pragma unroll
    for (int k = 0; k < IPT; ++k) {
      const uint32_t i = t + k * NT;
      probe[k] = false;
      walk[k] = false;
      if (i < I) {
        h0[k] = __ldg(hit0 + (uint64_t)s * I + i);
        tp0[k] = __ldg(tpf0 + (uint64_t)s * I + i);
        uint32_t p = h0[k];
        if ((int32_t)i == ja0 && jn0 > p) p = jn0;
        if ((int32_t)i == ja1 && jn1 > p) p = jn1;
        if ((int32_t)i == ja2 && jn2 > p) p = jn2;
        pos[k] = p;
        // s_end[i] != 0: the instance has window inserts visible to this row
        probe[k] = s_end[i] != 0u && p < nb;
        key[k] = probe[k] ? __ldg(hash + off + p) : 0ull;
      }
    }
    if (warp == 0) {
      // Wait until the inserts of jobs [done, need) are in: the leading run of done flags among the
      // next 32 is taken, and the first one not yet done is waited for.
      uint32_t f = s_done;
      bool abort = false;
      while ((int64_t)f < need && !abort) {
        const uint32_t x = f + (uint32_t)lane;
        const bool ok = (int64_t)x < need && psk::ld_acquire_u32(sync.done + x) != 0u;
        const unsigned okm = __ballot_sync(0xffffffffu, ok);
        const uint32_t nok = (okm == 0xffffffffu) ? 32u : (uint32_t)(__ffs(~okm) - 1);
        if (nok == 0u) {
          bool got = true;
          if (lane == 0) got = wait_flag(sync.done + f, err, sync.wait_ns);
          abort = !__shfl_sync(0xffffffffu, got, 0);
          continue;
        }
        f += nok;
      }
      if (lane == 0) {
        s_done = f;
        s_abort = abort ? 1 : 0;
      }
    }
    __syncthreads();
    if (s_abort) return;  // block-uniform
#pragma unroll
    for (int k = 0; k < IPT; ++k) {
      const uint32_t i = t + k * NT;
      if (probe[k] && psk::delta_contains(delta, nslots, i, key[k])) {
        walk[k] = true;
        s_res[i] = pos[k];
        s_walk[atomicAdd(&s_nwalk, 1u)] = i;
      }
    }
    __syncthreads();
    const uint32_t nwalk = s_nwalk;
    if (nwalk) {
      for (uint32_t x = warp; x < nwalk; x += NW) {
        const uint32_t i = s_walk[x];
        auto cached = [&](uint64_t k) { return k < nb && psk::delta_contains(delta, nslots, i, __ldg(hash + off + k)); };
        const uint64_t hnew = psk::warp_first_miss_search_hint((uint64_t)s_res[i] + 1, nb, s_end[i], cached);
        __syncwarp();
        if (lane == 0) s_res[i] = (uint32_t)hnew;
      }
      __syncthreads();
    }
    const uint32_t slot = s % psk::kHitSlots;
#pragma unroll
    for (int k = 0; k < IPT; ++k) {
      const uint32_t i = t + k * NT;
      if (i < I) {
        const uint32_t h = walk[k] ? s_res[i] : pos[k];
        sync.hitring[(uint64_t)slot * sync.ring_stride + i] = h;
        sync.tpfring[(uint64_t)slot * sync.ring_stride + i] = h == h0[k] ? tp0[k] : __uint_as_float(psk::kNoTpfBits);
      }
    }
    __syncthreads();
    if (t == 0) {
      s_nwalk = 0;
      __threadfence();  // the row's hits before its flag
      psk::st_release_u32(sync.ready + s, 1u);
    }
  }
}

// Deciding block.  Thread t < NTI owns instances t * IPT .. t * IPT + IPT - 1; thread 0 publishes
// the decisions.  The last warp only waits for the probe blocks' ready flags (thread NTI): an
// acquire load holds up its thread's later memory accesses, so that warp does nothing else.  Block
// reductions: each instance warp reduces its lanes with single-instruction warp reductions, writes
// one partial, and after the barrier every instance warp reduces the partials itself.
// Instance state is kept as padded structure-of-arrays in shared memory, so a thread reads its IPT
// consecutive instances' values of one field with one vector load; the capacity guard is one
// compare against the free KV room, stored as -1 where the decode-slot guard fails.
template <int N>
__device__ __forceinline__ void ld_u32v(const void* p, uint32_t (&v)[N]) {
  static_assert(N == 1 || N == 2 || N == 4, "vector of 1, 2 or 4");
  if (N == 1) {
    v[0] = *reinterpret_cast<const uint32_t*>(p);
  } else if (N == 2) {
    const uint2 x = *reinterpret_cast<const uint2*>(p);
    v[0] = x.x;
    v[N > 1 ? 1 : 0] = x.y;
  } else {
    const uint4 x = *reinterpret_cast<const uint4*>(p);
    v[0] = x.x;
    v[N > 1 ? 1 : 0] = x.y;
    v[N > 2 ? 2 : 0] = x.z;
    v[N > 3 ? 3 : 0] = x.w;
  }
}

template <int N>
__device__ __forceinline__ void st_zero_u32v(void* p) {
  if (N == 1) *reinterpret_cast<uint32_t*>(p) = 0u;
  else if (N == 2) *reinterpret_cast<uint2*>(p) = make_uint2(0u, 0u);
  else *reinterpret_cast<uint4*>(p) = make_uint4(0u, 0u, 0u, 0u);
}

template <int N>
__device__ __forceinline__ void ld_u64v(const void* p, uint64_t (&v)[N]) {
  if (N == 1) {
    v[0] = *reinterpret_cast<const unsigned long long*>(p);
  } else {
#pragma unroll
    for (int k = 0; k < N; k += 2) {
      const ulonglong2 x = reinterpret_cast<const ulonglong2*>(p)[k / 2];
      v[k] = x.x;
      v[k + 1 < N ? k + 1 : k] = x.y;
    }
  }
}

// q and S within [0, 2^30): with L, n < 2^30 the sums S + L and q + n are exact in 32 bits.
__device__ __forceinline__ bool narrow_qs(int64_t q, int64_t S) {
  return q >= 0 && q < (1ll << 30) && S >= 0 && S < (1ll << 30);
}

template <int IPT>
__device__ void decide_rows(const psk::RowPre* __restrict__ rows, uint32_t R, uint32_t I, psk::StateSoA committed,
                            psk::StateSoA pending, const psk::DevModel& m, int32_t* assign, uint8_t* __restrict__ path,
                            uint32_t* __restrict__ hit_chosen, uint32_t* err, const psk::GreedySync& sync,
                            unsigned long long* smem_raw) {
  const uint32_t Ip = sync.ring_stride;  // I rounded up to a multiple of 4
  // Every [Ip] array starts 16-byte aligned (Ip is a multiple of 4); the 8-byte arrays come first.
  int64_t* s_q = reinterpret_cast<int64_t*>(smem_raw);    // [Ip] queued prefill tokens
  int64_t* s_S = s_q + Ip;                                // [Ip] KV tokens held
  uint64_t* s_key0 = reinterpret_cast<uint64_t*>(s_S + Ip);  // [Ip] D-C-Q key bits of (b, qr) (psk::dcq_key0)
  int64_t* s_M = reinterpret_cast<int64_t*>(s_key0 + Ip);    // [Ip] KV capacity
  uint32_t* s_hit = reinterpret_cast<uint32_t*>(s_M + Ip);   // [4][Ip] probed hits of rows r .. r + 3
  uint32_t* s_tpf = s_hit + 4 * Ip;                          // [4][Ip] T_pf at those hits (bits)
  uint32_t* s_ovr = s_tpf + 4 * Ip;                          // [2][Ip] lcp raises for the next row
  int32_t* s_room = reinterpret_cast<int32_t*>(s_ovr + 2 * Ip);  // [Ip] free KV room, -1 if no slot
  float* s_dec0 = reinterpret_cast<float*>(s_room + Ip);     // [Ip] InstTerms, field by field
  float* s_f = s_dec0 + Ip;
  float* s_tq = s_f + Ip;
  int32_t* s_Bp = reinterpret_cast<int32_t*>(s_tq + Ip);
  int32_t* s_b = s_Bp + Ip;                                  // [Ip] decoding requests
  int32_t* s_qr = s_b + Ip;                                  // [Ip] queued requests
  int32_t* s_Bmax = s_qr + Ip;                               // [Ip] decode-slot limit
  __shared__ psk::RowPre s_row[8];  // rows r .. r + kRingAhead (a ring of 8 so no reader is overtaken)
  __shared__ int s_wide;            // some instance's q or S left [0, 2^30): 64-bit token sums from then on
  __shared__ int32_t s_jm[16];      // pick of request x in s_jm[x & 15] (-1: rejected)
  __shared__ uint32_t s_red_w[32];  // per-warp W_min (order-preserving bits)
  __shared__ uint4 s_red_k[32];     // per-warp pick: key (x, y), instance (z), hit (w)

  const int t = threadIdx.x;
  const int NT = blockDim.x;
  const int NTI = NT - 32;
  const bool sig = t == NTI;
  const int lane = t & 31;
  const int warp = t >> 5;
  const int NWI = NTI >> 5;               // instance warps
  const uint32_t i0 = (uint32_t)t * IPT;  // first owned instance (>= I for the signalling warp)
  const bool owner = t < NTI;             // false for the whole signalling warp
  const bool has = owner && i0 < I;       // the thread owns instances (then i0 + IPT <= Ip)
  // instance terms of i after a state change (decode-slot guard folded into the KV room)
  auto set_terms = [&](uint32_t i) {
    const psk::InstTerms it = psk::inst_terms(m, s_b[i], s_qr[i], s_q[i], s_Bmax[i]);
    s_dec0[i] = it.dec0;
    s_f[i] = it.f;
    s_tq[i] = it.tq;
    s_Bp[i] = it.Bp;
    s_room[i] = it.okB ? psk::kv_room(s_S[i], s_M[i]) : -1;
    s_key0[i] = psk::dcq_key0(s_b[i], s_qr[i]);
  };

  if (t == 0) s_wide = 0;
  __syncthreads();
  for (uint32_t i = t; i < Ip; i += NT) {
    if (i < I) {
      s_b[i] = committed.b[i];
      s_qr[i] = committed.qr[i];
      s_q[i] = committed.q[i];
      s_S[i] = committed.S[i];
      s_M[i] = committed.M[i];
      s_Bmax[i] = committed.Bmax[i];
      set_terms(i);
      if (!narrow_qs(s_q[i], s_S[i])) s_wide = 1;
    } else {
      s_room[i] = -1;  // padding: never capacity-eligible
    }
  }
  for (uint32_t i = t; i < 2 * Ip; i += NT) s_ovr[i] = 0u;
  if (t < 16) s_jm[t] = -1;
  if (t < kRingAhead * psk::kRowWords) {  // rows 0 .. kRingAhead - 1
    const uint32_t rr = (uint32_t)(t / psk::kRowWords);
    if (rr < R)
      reinterpret_cast<uint4*>(&s_row[rr])[t % psk::kRowWords] =
          __ldg(reinterpret_cast<const uint4*>(rows + rr) + (t % psk::kRowWords));
  }
  bool timed_out = false;
  if (sig) {
    for (uint32_t x = 0; x < 2 && x < R && !timed_out; ++x) timed_out = !wait_flag(sync.ready + x, err, sync.wait_ns);
  }
  __syncthreads();
  // hits of rows 0 and 1, one copy group each (each thread copies and later reads only its own)
  static_assert(IPT == 1 || IPT == 2 || IPT == 4, "one 4-, 8- or 16-byte copy per array and row");
  auto copy_row = [&](uint32_t x) {
    if (has) {
      const uint64_t src = (uint64_t)(x % psk::kHitSlots) * Ip + i0;
      const uint32_t dst = (x & 3u) * Ip + i0;
      psk::cp_async_bytes<4 * IPT>(s_hit + dst, sync.hitring + src);
      psk::cp_async_bytes<4 * IPT>(s_tpf + dst, sync.tpfring + src);
    }
  };
  if (R > 0) copy_row(0);
  psk::cp_async_commit();
  if (R > 1) copy_row(1);
  psk::cp_async_commit();

  int32_t jprev = -1;  // pick of request r - 1
  uint32_t hr[IPT];

  for (uint32_t r = 0; r < R; ++r) {
    if (!owner) {  // the signalling warp: row r + 2's ready flag, then the step's two barriers
      uint32_t ready_seen = 1u;
      if (sig && r + 2 < R && !timed_out) ready_seen = psk::ld_acquire_u32(sync.ready + r + 2);
      __syncthreads();  // (C)
      if (sig && ready_seen == 0u) timed_out = !wait_flag(sync.ready + r + 2, err, sync.wait_ns);
      __syncthreads();  // (D)
      continue;
    }
    const psk::RowPre& cur = s_row[r & 7];
    // ---- P0: row-constant refill, row r's hits, pass 1 ------------------------------------------
    if (t < psk::kRowWords && r + kRingAhead < R)
      psk::cp_async16(reinterpret_cast<uint4*>(&s_row[(r + kRingAhead) & 7]) + t,
                      reinterpret_cast<const uint4*>(rows + r + kRingAhead) + t);
    psk::cp_async_wait_group<1>();  // this thread's copies of row r (and row constants <= r + 4)
    const psk::RowConst rc = row_of(cur);
    const bool narrow = s_wide == 0;  // a thread owning an instance that left the range set the flag itself
    const uint32_t lcp0 = cur.lcp[0];
    float Wk[IPT], tpk[IPT];
    bool inA[IPT];
    uint32_t wbest = 0xFFFFFFFFu;  // order-preserving bits of this thread's W_min over A
    if (has) {
      uint32_t hb[IPT], ov[IPT], tb[IPT], rm[IPT];
      ld_u32v<IPT>(s_hit + (r & 3u) * Ip + i0, hb);
      ld_u32v<IPT>(s_tpf + (r & 3u) * Ip + i0, tb);
      uint32_t* op = s_ovr + (r & 1u) * Ip + i0;
      ld_u32v<IPT>(op, ov);
      ld_u32v<IPT>(s_room + i0, rm);
      uint32_t anyov = 0u;
#pragma unroll
      for (int k = 0; k < IPT; ++k) anyov |= ov[k];
      if (anyov) st_zero_u32v<IPT>(op);
#pragma unroll
      for (int k = 0; k < IPT; ++k) {
        uint32_t h = hb[k] > ov[k] ? hb[k] : ov[k];
        if ((int32_t)(i0 + k) == jprev && lcp0 > h) h = lcp0;
        hr[k] = h;
        // T_pf at the hit: the ring's value unless it is marked unknown (the probe blocks raised the
        // hit) or the hit was raised here; W = T_pf(n, c) - T_pf(0, L)
        tpk[k] = (h == hb[k] && tb[k] != psk::kNoTpfBits) ? __uint_as_float(tb[k]) : psk::t_pf32(m, rc.L, h);
        Wk[k] = __fsub_rn(tpk[k], rc.t_cached);
        inA[k] = (int32_t)rc.L <= (int32_t)rm[k];
        if (inA[k]) wbest = min(wbest, psk::f2ord(Wk[k]));
      }
    } else {
#pragma unroll
      for (int k = 0; k < IPT; ++k) inA[k] = false;
    }
    wbest = __reduce_min_sync(0xffffffffu, wbest);
    if (lane == 0) s_red_w[warp] = wbest;
    __syncthreads();  // (C)

    // ---- P1: W_min, pass 2, the row's argmin; lcp raises for row r + 1 --------------------------
    const uint32_t wmin_o = __reduce_min_sync(0xffffffffu, lane < NWI ? s_red_w[lane] : 0xFFFFFFFFu);
    const bool anyA = wmin_o != 0xFFFFFFFFu;  // a W of a pair in A never maps to all ones (not NaN)
    const float wmin = psk::ord2f(wmin_o);
    uint64_t bkey = psk::kNoKey;
    uint32_t btie = 0xFFFFFFFFu, bh = 0u;
    bool inC[IPT];
    bool anyC = false;
#pragma unroll
    for (int k = 0; k < IPT; ++k) {
      inC[k] = inA[k] && psk::pair_in_c(rc, Wk[k], wmin);
      anyC |= inC[k];
    }
    if (anyC) {
      uint32_t dec0[IPT], fe[IPT], tq[IPT], Bp[IPT];
      uint64_t q[IPT], S[IPT], k0[IPT];
      ld_u32v<IPT>(s_dec0 + i0, dec0);
      ld_u32v<IPT>(s_f + i0, fe);
      ld_u32v<IPT>(s_tq + i0, tq);
      ld_u32v<IPT>(s_Bp + i0, Bp);
      ld_u64v<IPT>(s_q + i0, q);
      ld_u64v<IPT>(s_S + i0, S);
      ld_u64v<IPT>(s_key0 + i0, k0);
#pragma unroll
      for (int k = 0; k < IPT; ++k) {
        if (!inC[k]) continue;
        psk::InstTerms it;
        it.dec0 = __uint_as_float(dec0[k]);
        it.f = __uint_as_float(fe[k]);
        it.tq = __uint_as_float(tq[k]);
        it.Bp = (int32_t)Bp[k];
        it.okB = 1;
        psk::PairW x;
        x.W = Wk[k];
        x.tpf = tpk[k];
        x.n = (int64_t)rc.L - 16 * (int64_t)hr[k];
        x.inA = true;
        float tpot, ttft;
        if (narrow)
          psk::pair_lat32(m, rc, x.tpf, (int32_t)x.n, it.dec0, it.f, it.tq, it.Bp, (int32_t)q[k], (int32_t)S[k], &tpot,
                          &ttft);
        else
          psk::pair_lat(m, rc, x, it, (int64_t)q[k], (int64_t)S[k], &tpot, &ttft);
        uint64_t key;
        uint32_t tie = i0 + k;
        if (psk::pair_admitted(m, rc, tpot, ttft)) {
          key = psk::packed_key(0u, psk::value_in_t(m, psk::key0_from_dcq(m, k0[k]), hr[k], tpot, rc.tpot_target));
          if (m.sel == psk::kSelHCQ) tie = psk::tie_in_t(m, i0 + k, (int32_t)(k0[k] & 0x3FFFFull));
        } else {
          key = psk::packed_key(1u, psk::value_fallback(m, (uint64_t)q[k] + (uint64_t)x.n, (uint32_t)Bp[k], k0[k], hr[k]));
        }
        if (key < bkey || (key == bkey && tie < btie)) {
          bkey = key;
          btie = tie;
          bh = hr[k];
        }
      }
    }
    {
      uint64_t wk;
      uint32_t wi, wh;
      psk::warp_pick_min(bkey, btie, bh, &wk, &wi, &wh);
      if (lane == 0) s_red_k[warp] = make_uint4((uint32_t)wk, (uint32_t)(wk >> 32), wi, wh);
    }
    // Row r + 1's raises from requests r - 1 .. r - kLag + 1 (thread d - 1 takes request r - d); the
    // raise from request r itself is applied in registers next step.
    if (t < psk::kLcpBack - 1 && r + 1 < R) {
      const uint32_t d = (uint32_t)t + 1u;
      const int32_t jd = r >= d ? s_jm[(r - d) & 15u] : -1;
      const uint32_t v = s_row[(r + 1) & 7].lcp[d];
      if (jd >= 0 && v > 0u) atomicMax(s_ovr + ((r + 1) & 1u) * Ip + (uint32_t)jd, v);
    }
    __syncthreads();  // (D)

    // ---- P2: the pick, its state, its insert job; copies of row r + 2 ----------------------------
    uint64_t key;
    uint32_t j, hj;
    {
      const uint4 pk = lane < NWI ? s_red_k[lane] : make_uint4(0xFFFFFFFFu, 0xFFFFFFFFu, 0xFFFFFFFFu, 0u);
      psk::warp_pick_min(((uint64_t)pk.y << 32) | pk.x, pk.z, pk.w, &key, &j, &hj);
      j &= psk::kTieInstMask;
    }
    const bool pick = anyA && key != psk::kNoKey;
    if (!pick) hj = 0u;
    if (t == 0) {
      assign[r] = pick ? (int32_t)j : -1;
      path[r] = pick ? (uint8_t)(key >> 62) : (uint8_t)2;
      hit_chosen[r] = hj;
      s_jm[r & 15u] = pick ? (int32_t)j : -1;
      psk::st_relaxed_u64(sync.jobs + r, kJobValid | ((unsigned long long)hj << 32) | (pick ? j : 0xFFFFFFFFu));
    }
    if (pick && j >= i0 && j < i0 + IPT) {
      s_qr[j] += 1;
      s_q[j] += (int64_t)rc.L - 16 * (int64_t)hj;
      s_S[j] += (int64_t)rc.L;
      set_terms(j);
      if (!narrow_qs(s_q[j], s_S[j])) s_wide = 1;  // seen from the next step on (after its barriers)
    }
    if (r + 2 < R) copy_row(r + 2);
    psk::cp_async_commit();
    jprev = pick ? (int32_t)j : -1;
  }
  psk::cp_async_wait_all();
  __syncthreads();
  for (uint32_t i = t; i < I; i += NT) {
    pending.b[i] = s_b[i];
    pending.qr[i] = s_qr[i];
    pending.q[i] = s_q[i];
    pending.S[i] = s_S[i];
    pending.M[i] = s_M[i];
    pending.Bmax[i] = s_Bmax[i];
  }
}

template <int IPT>
__global__ void __launch_bounds__(544, 1)
greedy_pipe_kernel(const psk::RowPre* __restrict__ rows, const uint64_t* __restrict__ hash, uint32_t R, uint32_t I,
                   const uint32_t* __restrict__ hit0, const float* __restrict__ tpf0, psk::StateSoA committed,
                   psk::StateSoA pending, psk::DevModel m, psk::DeltaSlot* delta, uint64_t nslots, int32_t* assign,
                   uint8_t* __restrict__ path, uint32_t* __restrict__ hit_chosen, uint32_t* err, psk::GreedySync sync) {
  extern __shared__ unsigned long long smem_raw[];
  if (blockIdx.x == 0) {
    decide_rows<IPT>(rows, R, I, committed, pending, m, assign, path, hit_chosen, err, sync, smem_raw);
  } else if (blockIdx.x <= kInsertBlocks) {
    insert_blocks(rows, hash, R, delta, nslots, err, sync);
  } else {
    probe_rows<IPT>(rows, hash, R, I, hit0, tpf0, delta, nslots, err, sync, smem_raw);
  }
}

size_t greedy_pipe_smem(uint32_t I, uint32_t Ip) {
  // 4 eight-byte and 18 four-byte [Ip] arrays (q, S, key0, M; hit and T_pf rings, raises, room,
  // dec0, f, tq, Bp, b, qr, B_max)
  const size_t decide = (size_t)Ip * (4 * sizeof(int64_t) + 18 * sizeof(uint32_t));
  const size_t probe = (size_t)I * 3 * sizeof(uint32_t);
  return decide > probe ? decide : probe;
}

template <int IPT>
cudaError_t greedy_pipe_launch(const psk::RowPre* rows, const psk::WindowDev& w, uint32_t I, const uint32_t* hit0,
                               const float* tpf0, psk::StateSoA committed, psk::StateSoA pending, const psk::DevModel& m,
                               psk::DeltaSlot* delta, uint64_t nslots, int32_t* assign, uint8_t* path,
                               uint32_t* hit_chosen, uint32_t* err, const psk::GreedySync& sync, uint32_t nt,
                               cudaStream_t s) {
  const size_t smem = greedy_pipe_smem(I, sync.ring_stride);
  cudaError_t e = cudaFuncSetAttribute(greedy_pipe_kernel<IPT>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (e != cudaSuccess) return e;
  const uint64_t* hash = w.hash;
  uint32_t R = w.R;
  psk::StateSoA c = committed, p = pending;
  psk::DevModel mm = m;
  psk::GreedySync sy = sync;
  void* args[] = {(void*)&rows, (void*)&hash, (void*)&R, (void*)&I, (void*)&hit0, (void*)&tpf0, (void*)&c, (void*)&p,
                  (void*)&mm, (void*)&delta, (void*)&nslots, (void*)&assign, (void*)&path, (void*)&hit_chosen,
                  (void*)&err, (void*)&sy};
  // all blocks must be resident at once: they wait on one another
  return cudaLaunchCooperativeKernel((const void*)greedy_pipe_kernel<IPT>, dim3(1 + kInsertBlocks + kProbeBlocks),
                                     dim3(nt), args, smem, s);
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
  if (w.R == 0) return cudaSuccess;
  cudaError_t e = cudaMemsetAsync(sync.done, 0, (size_t)w.R * sizeof(uint32_t), s);
  if (e == cudaSuccess) e = cudaMemsetAsync(sync.ready, 0, (size_t)w.R * sizeof(uint32_t), s);
  if (e == cudaSuccess) e = cudaMemsetAsync(sync.jobs, 0, (size_t)w.R * sizeof(unsigned long long), s);
  if (e != cudaSuccess) return e;
  // up to 512 threads each owning IPT consecutive instances (IPT = 1, 2 or 4 for I up to 2048),
  // plus one signalling warp
  const uint32_t ipt = I <= 512 ? 1u : (I <= 1024 ? 2u : 4u);
  const uint32_t nt = ((I + ipt - 1) / ipt + 31) / 32 * 32 + 32;
#define PS_GREEDY_P(IPT)                                                                                      \
  return greedy_pipe_launch<IPT>(rows, w, I, hit0, tpf0, committed, pending, m, delta, delta_nslots, assign, path, \
                                 hit_chosen, err, sync, nt, s)
  if (ipt == 1) PS_GREEDY_P(1);
  if (ipt == 2) PS_GREEDY_P(2);
  if (ipt == 4 && I <= 2048) PS_GREEDY_P(4);
#undef PS_GREEDY_P
  return cudaErrorInvalidValue;
}

// The delta table only holds one window's blocks: clear it whole after each window.
cudaError_t launch_delta_clear(psk::DeltaSlot* delta, uint64_t nslots, cudaStream_t s) {
  return cudaMemsetAsync(delta, 0, nslots * sizeof(psk::DeltaSlot), s);
}

}  // namespace pskl
