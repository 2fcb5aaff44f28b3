// Greedy in-window assignment (Algorithm 1 applied to the window's requests in arrival order).
//
// The paper's gateway decides each request online and updates the instance records along the
// request path before the next decision (Section 4, Metadata service; Section 7).  Two kernels
// replay that sequence for a whole window on the GPU:
//   greedy_kernel       any cache (the probe's linear mode), described here;
//   greedy_pipe_kernel  prefix-closed caches (the search mode), a pipelined cooperative launch of
//                       deciding, insert, probe and summary blocks, described at its section below.
// greedy_kernel is one persistent thread block whose threads each own up to IPT instances.  Per
// request r:
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
// Prefix-closed caches (the probe's search mode): a pipelined greedy pass over four kinds of
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
//   Deciding block (block 0).  A feeder warp stages each row's summary, row constants and probed
//   hits in shared memory; the deciding warp decides the requests in arrival order from the
//   summaries, correcting them for the last kSpecLag picks (the lag-d speculation below), updates
//   the pick's state and publishes each decision as an insert job.  No table access is on its
//   per-request path.
//   Insert blocks.  Groups of kInsertGroup blocks take the jobs round-robin; a group's members split
//   each job's chain blocks chain[h, nb) between them, insert them into delta_j and count the job done.
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
//   Summary blocks.  Take the rows round-robin; evaluate row s on every instance against the state
//   before decision s - kSpecLag and publish its summary (below).
// Every cross-block wait is bounded (GreedySync::wait_ns, 1 s unless the caller set another limit);
// on expiry the waiter records PS_ERR_TIMEOUT and stops waiting, so the launch always ends.  Each
// role keeps the instance state it needs in its own shared memory.

constexpr uint32_t kInsertBlocks = 16;   // insert blocks
constexpr uint32_t kProbeBlocks = 16;    // probe blocks
constexpr uint32_t kSummaryBlocks = 32;  // summary blocks (lag-d speculation, below)
constexpr uint32_t kPipeThreads = 256;   // threads of every block of the launch
constexpr uint32_t kFeedRing = 4;        // rows staged in the deciding block's shared memory
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

// Bounded spin until *count >= want (acquire).  false after limit_ns (and the error bit is set).
__device__ __forceinline__ bool wait_count(const uint32_t* count, uint32_t want, uint32_t* err, uint64_t limit_ns) {
  if (psk::ld_acquire_u32(count) >= want) return true;
  const uint64_t t0 = psk::globaltimer_ns();
  while (psk::ld_acquire_u32(count) < want) {
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

// Insert blocks, in groups of kInsertGroup: group g inserts the chain tails of jobs g, g + the number
// of groups, ...; the group's members split a tail by position (member m takes positions
// h + m * 256 + t, stride kInsertGroup * 256) and each adds 1 to the job's done count once its
// inserts are in, so the job's blocks are all in when the count reaches kInsertGroup.  A thread
// claims the home slots of kInsertBatch keys at once (the claims are independent) and follows the
// rare occupied home slot on its own.
constexpr uint32_t kInsertGroup = 4;
constexpr int kInsertBatch = 4;
static_assert(kInsertBlocks % kInsertGroup == 0, "whole insert groups");

__device__ __forceinline__ void insert_tail(psk::DeltaSlot* delta, uint64_t nslots, uint32_t j,
                                            const uint64_t* __restrict__ chain, uint64_t first, uint64_t nb,
                                            uint64_t stride, uint32_t* err) {
  for (uint64_t p0 = first; p0 < nb; p0 += kInsertBatch * stride) {
    uint64_t key[kInsertBatch], slot[kInsertBatch];
    unsigned long long old[kInsertBatch];
#pragma unroll
    for (int q = 0; q < kInsertBatch; ++q) {
      const uint64_t p = p0 + (uint64_t)q * stride;
      key[q] = p < nb ? __ldg(chain + p) : psk::kEmpty;
    }
#pragma unroll
    for (int q = 0; q < kInsertBatch; ++q) {
      old[q] = ~0ull;
      if (key[q] != psk::kEmpty && key[q] != psk::kTomb) {
        slot[q] = psk::delta_home(key[q], nslots);
        old[q] = atomicCAS(&delta[slot[q]].hash, psk::kEmpty, (unsigned long long)key[q]);
      }
    }
#pragma unroll
    for (int q = 0; q < kInsertBatch; ++q) {
      if (key[q] == psk::kEmpty || key[q] == psk::kTomb) continue;
      if (old[q] == psk::kEmpty) {
        __stcg(&delta[slot[q]].tag, j + 1);
      } else if (!psk::delta_insert_from(delta, nslots, j, key[q], psk::delta_next(slot[q], nslots))) {
        atomicOr(err, psk::kErrDeltaFull);
      }
    }
  }
}

__device__ void insert_blocks(const psk::RowPre* __restrict__ rows, const uint64_t* __restrict__ hash, uint32_t R,
                              psk::DeltaSlot* delta, uint64_t nslots, uint32_t* err, const psk::GreedySync& sync) {
  __shared__ unsigned long long s_job;
  const uint32_t t = threadIdx.x;
  const uint32_t ib = blockIdx.x - 1;
  const uint32_t group = ib / kInsertGroup, member = ib % kInsertGroup;
  constexpr uint32_t kGroups = kInsertBlocks / kInsertGroup;
  for (uint32_t job = group; job < R; job += kGroups) {
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
      insert_tail(delta, nslots, j, hash + off, (uint64_t)hj + member * blockDim.x + t, nb,
                  (uint64_t)kInsertGroup * blockDim.x, err);
    }
    __syncthreads();
    if (t == 0) {
      __threadfence();  // every thread's inserts before the count
      atomicAdd(sync.done + job, 1u);
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
  unsigned long long cyc_done = 0;  // thread 0: cycles spent waiting for inserts
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
      const long long c0 = clock64();
      uint32_t f = s_done;
      bool abort = false;
      while ((int64_t)f < need && !abort) {
        const uint32_t x = f + (uint32_t)lane;
        const bool ok = (int64_t)x < need && psk::ld_acquire_u32(sync.done + x) >= kInsertGroup;
        const unsigned okm = __ballot_sync(0xffffffffu, ok);
        const uint32_t nok = (okm == 0xffffffffu) ? 32u : (uint32_t)(__ffs(~okm) - 1);
        if (nok == 0u) {
          bool got = true;
          if (lane == 0) got = wait_count(sync.done + f, kInsertGroup, err, sync.wait_ns);
          abort = !__shfl_sync(0xffffffffu, got, 0);
          continue;
        }
        f += nok;
      }
      if (lane == 0) {
        s_done = f;
        s_abort = abort ? 1 : 0;
        cyc_done += (unsigned long long)(clock64() - c0);
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
  if (t == 0 && sync.stats) atomicAdd(sync.stats + psk::kGsProbeDoneWait, cyc_done);
}

// q and S within [0, 2^30): with L, n < 2^30 the sums S + L and q + n are exact in 32 bits.
__device__ __forceinline__ bool narrow_qs(int64_t q, int64_t S) {
  return q >= 0 && q < (1ll << 30) && S >= 0 && S < (1ll << 30);
}

// ---- lag-d speculation: summary blocks and the deciding warp ------------------------------------
//
// Row s's decision depends on the state left by decisions 0 .. s - 1.  Summary blocks evaluate row s
// on every instance against the state before decision s - kSpecLag (replaying the published jobs
// into their own copy of the state), and publish per warp the kKeysPerWarp smallest (packed key, tie)
// pairs of C with their W and hit, and the kWPerWarp smallest W of A, with the bounds of what they
// did not publish (RowSummary).  Only the instances picked by decisions s - kSpecLag .. s - 1 (the
// touched ones) have changed since: their state, and their caches (each touched instance's hit on
// row s rises to the common prefix with the requests it took).  Every other instance keeps its
// capacity test, W and key.  So the deciding warp re-evaluates the touched instances only, and:
//   * W_min over A is the smaller of the touched instances' W and the smallest published W of an
//     untouched instance, known exactly when that W lies at or below the W bound;
//   * in-window inserts only lengthen hits, so W_min can only fall unless an instance leaves A; if
//     it rose above the summary's W_min, the summary's C may miss members (full pass);
//   * with W_min at or below the summary's, C of the current state holds no untouched pair outside
//     the summary's C, and a published untouched pair stays in C when W - W_min <= eta Z still holds;
//   * the pick is the smallest (key, tie) over the surviving published pairs and the touched pairs
//     in C; every unpublished pair has (key, tie) >= the key bound, so a pick below the bound is
//     exact.
// Otherwise (W_min unknown or risen, or no pick below the bound) the warp evaluates the whole row on
// the current state.  Both ways give Algorithm 1's decision exactly.
//
// Deciding block: warp 0 decides, warp 1 (the feeder) copies each row's summary, row constants, hits
// and T_pf into a shared-memory ring as soon as the summary is published; the two hand off through
// shared-memory counters (the feeder's row count, the decider's consumed count), each wait bounded.

static_assert(kPipeThreads == 32 * psk::kSumWarps, "a summary block is kSumWarps warps");

// Instance state of the summary blocks and the deciding warp: padded structure-of-arrays in shared
// memory, [Ip] each, 8-byte arrays first (64 bytes per instance).
struct InstSmem {
  int64_t* q;
  int64_t* S;
  int64_t* M;
  uint64_t* kd;   // D-C-Q key bits of (b, qr) (psk::dcq_key0)
  int32_t* room;  // free KV room, -1 when the decode-slot guard fails
  float* dec0;
  float* f;
  float* tq;
  int32_t* Bp;
  int32_t* b;
  int32_t* qr;
  int32_t* Bmax;
};
constexpr size_t kInstSmemBytes = 4 * sizeof(int64_t) + 8 * sizeof(int32_t);

__device__ __forceinline__ InstSmem inst_smem(unsigned long long* raw, uint32_t Ip) {
  InstSmem a;
  a.q = reinterpret_cast<int64_t*>(raw);
  a.S = a.q + Ip;
  a.M = a.S + Ip;
  a.kd = reinterpret_cast<uint64_t*>(a.M + Ip);
  a.room = reinterpret_cast<int32_t*>(a.kd + Ip);
  a.dec0 = reinterpret_cast<float*>(a.room + Ip);
  a.f = a.dec0 + Ip;
  a.tq = a.f + Ip;
  a.Bp = reinterpret_cast<int32_t*>(a.tq + Ip);
  a.b = a.Bp + Ip;
  a.qr = a.b + Ip;
  a.Bmax = a.qr + Ip;
  return a;
}

// Derived terms of instance i after a state change (the decode-slot guard folded into the KV room).
__device__ __forceinline__ void inst_refresh(const InstSmem& a, const psk::DevModel& m, uint32_t i) {
  const psk::InstTerms it = psk::inst_terms(m, a.b[i], a.qr[i], a.q[i], a.Bmax[i]);
  a.dec0[i] = it.dec0;
  a.f[i] = it.f;
  a.tq[i] = it.tq;
  a.Bp[i] = it.Bp;
  a.room[i] = it.okB ? psk::kv_room(a.S[i], a.M[i]) : -1;
  a.kd[i] = psk::dcq_key0(a.b[i], a.qr[i]);
}

__device__ __forceinline__ void inst_load(const InstSmem& a, const psk::StateSoA& st, const psk::DevModel& m,
                                          uint32_t i) {
  a.b[i] = st.b[i];
  a.qr[i] = st.qr[i];
  a.q[i] = st.q[i];
  a.S[i] = st.S[i];
  a.M[i] = st.M[i];
  a.Bmax[i] = st.Bmax[i];
  inst_refresh(a, m, i);
}

// The values of one instance's state a pair evaluation reads.
struct InstVals {
  int64_t q, S;
  uint64_t kd;  // dcq_key0(b, qr)
  int32_t room;
  float dec0, f, tq;
  int32_t Bp;
};

__device__ __forceinline__ InstVals inst_vals(const InstSmem& a, uint32_t i) {
  InstVals v;
  v.q = a.q[i];
  v.S = a.S[i];
  v.kd = a.kd[i];
  v.room = a.room[i];
  v.dec0 = a.dec0[i];
  v.f = a.f[i];
  v.tq = a.tq[i];
  v.Bp = a.Bp[i];
  return v;
}

// Instance i's state after it takes a request of L tokens at hit h (qr + 1, q + L - 16 h, S + L), as
// the state update of a decision computes it.
__device__ __forceinline__ InstVals inst_vals_after(const InstSmem& a, const psk::DevModel& m, uint32_t i, uint32_t L,
                                                    uint32_t h, int32_t* qr_out) {
  const int32_t qr = a.qr[i] + 1;
  InstVals v;
  v.q = a.q[i] + (int64_t)L - 16 * (int64_t)h;
  v.S = a.S[i] + (int64_t)L;
  const psk::InstTerms it = psk::inst_terms(m, a.b[i], qr, v.q, a.Bmax[i]);
  v.dec0 = it.dec0;
  v.f = it.f;
  v.tq = it.tq;
  v.Bp = it.Bp;
  v.room = it.okB ? psk::kv_room(v.S, a.M[i]) : -1;
  v.kd = psk::dcq_key0(a.b[i], qr);
  *qr_out = qr;
  return v;
}

__device__ __forceinline__ void inst_store(const InstSmem& a, uint32_t i, int32_t qr, const InstVals& v) {
  a.qr[i] = qr;
  a.q[i] = v.q;
  a.S[i] = v.S;
  a.kd[i] = v.kd;
  a.room[i] = v.room;
  a.dec0[i] = v.dec0;
  a.f[i] = v.f;
  a.tq[i] = v.tq;
  a.Bp[i] = v.Bp;
}

// One pair (row, instance i at hit h) on state v: W, the capacity guard, and the packed key and tie
// word the pair has in C (class 0 if the SLO admission passes, class 1 otherwise); key kNoKey
// outside A.  tpf_bits: T_pf at h if known, else kNoTpfBits.
struct PairKey {
  float W;
  uint64_t key;
  uint32_t tie;
  bool inA;
};

__device__ __forceinline__ PairKey pair_key_v(const psk::DevModel& m, const psk::RowConst& rc, const InstVals& v,
                                              uint32_t i, uint32_t h, uint32_t tpf_bits) {
  PairKey p;
  const float tpf = tpf_bits != psk::kNoTpfBits ? __uint_as_float(tpf_bits) : psk::t_pf32(m, rc.L, h);
  p.W = __fsub_rn(tpf, rc.t_cached);
  p.inA = (int32_t)rc.L <= v.room;
  p.key = psk::kNoKey;
  p.tie = i;
  if (p.inA) {
    const int32_t n = (int32_t)rc.L - (int32_t)(h << 4);
    float tpot, ttft;
    if (narrow_qs(v.q, v.S)) {
      psk::pair_lat32(m, rc, tpf, n, v.dec0, v.f, v.tq, v.Bp, (int32_t)v.q, (int32_t)v.S, &tpot, &ttft);
    } else {
      psk::InstTerms it;
      it.dec0 = v.dec0;
      it.f = v.f;
      it.tq = v.tq;
      it.Bp = v.Bp;
      it.okB = 1;
      psk::PairW x;
      x.W = p.W;
      x.tpf = tpf;
      x.n = n;
      x.inA = true;
      psk::pair_lat(m, rc, x, it, v.q, v.S, &tpot, &ttft);
    }
    if (psk::pair_admitted(m, rc, tpot, ttft)) {
      p.key = psk::packed_key(0u, psk::value_in_t(m, psk::key0_from_dcq(m, v.kd), h, tpot, rc.tpot_target));
      if (m.sel == psk::kSelHCQ) p.tie |= (uint32_t)(v.kd & 0x3FFFFull) << 12;
    } else {
      p.key = psk::packed_key(1u, psk::value_fallback(m, (uint64_t)v.q + (uint64_t)n, (uint32_t)v.Bp, v.kd, h));
    }
  }
  return p;
}

__device__ __forceinline__ PairKey pair_key_of(const psk::DevModel& m, const psk::RowConst& rc, const InstSmem& a,
                                               uint32_t i, uint32_t h, uint32_t tpf_bits) {
  return pair_key_v(m, rc, inst_vals(a, i), i, h, tpf_bits);
}

__device__ __forceinline__ bool kt_less(uint64_t k1, uint32_t t1, uint64_t k2, uint32_t t2) {
  return k1 < k2 || (k1 == k2 && t1 < t2);
}

// Warp minimum of a 64-bit word with single-instruction reductions on each half.
__device__ __forceinline__ unsigned long long warp_min_u64w(unsigned long long v) {
  const uint32_t hi = (uint32_t)(v >> 32);
  const uint32_t mhi = __reduce_min_sync(0xffffffffu, hi);
  const uint32_t mlo = __reduce_min_sync(0xffffffffu, hi == mhi ? (uint32_t)v : 0xFFFFFFFFu);
  return ((unsigned long long)mhi << 32) | mlo;
}

using psk::wait_smem_at_least;

// Summary block sb: rows sb, sb + kSummaryBlocks, ...  Thread t holds instances t, t + 256, ...
template <int IPT>
__device__ void summary_rows(const psk::RowPre* __restrict__ rows, uint32_t R, uint32_t I, psk::StateSoA committed,
                             const psk::DevModel& m, uint32_t* err, const psk::GreedySync& sync, uint32_t sb,
                             unsigned long long* smem_raw) {
  const uint32_t Ip = sync.ring_stride;
  const InstSmem a = inst_smem(smem_raw, Ip);
  __shared__ psk::RowPre s_row;
  __shared__ int32_t s_jm[16];  // pick of request x in s_jm[x & 15] (-1: rejected)
  static_assert(psk::kLcpBack <= psk::kSpecLag + 16, "the ring holds the picks the row's raises need");
  __shared__ uint32_t s_wmin[psk::kSumWarps];
  __shared__ uint32_t s_wb[psk::kSumWarps];
  __shared__ unsigned long long s_kb[psk::kSumWarps];
  __shared__ uint32_t s_tb[psk::kSumWarps];
  __shared__ int s_abort;
  const uint32_t t = threadIdx.x;
  const int lane = (int)(t & 31u), warp = (int)(t >> 5);
  for (uint32_t i = t; i < I; i += kPipeThreads) inst_load(a, committed, m, i);
  if (t < 16) s_jm[t] = -1;
  if (t == 0) s_abort = 0;
  uint32_t applied = 0;  // decisions [0, applied) are in this block's state
  unsigned long long cyc_job = 0, cyc_ready = 0, cyc_eval = 0;
  __syncthreads();
  for (uint32_t s = sb; s < R; s += kSummaryBlocks) {
    const int64_t need = (int64_t)s - psk::kSpecLag;  // decisions [0, need) count for row s
    const long long c0 = clock64();
    long long c1 = c0;
    // Each warp waits for the row's probed hits and loads its threads' hits and T_pf right away, so
    // the loads are in flight while warp 0 replays the decisions the row must see.
    const uint32_t slot = s % psk::kHitSlots;
    uint32_t hl[IPT], tl[IPT];
    {
      bool rdy = true;
      if (lane == 0) {
        rdy = wait_flag(sync.ready + s, err, sync.wait_ns);
        if (!rdy) s_abort = 1;
      }
      rdy = __shfl_sync(0xffffffffu, rdy ? 1 : 0, 0) != 0;
#pragma unroll
      for (int k = 0; k < IPT; ++k) {
        const uint32_t i = t + (uint32_t)k * kPipeThreads;
        hl[k] = 0u;
        tl[k] = psk::kNoTpfBits;
        if (rdy && i < I) {
          hl[k] = __ldcg(sync.hitring + (uint64_t)slot * Ip + i);
          tl[k] = __float_as_uint(__ldcg(sync.tpfring + (uint64_t)slot * Ip + i));
        }
      }
    }
    if (warp == 0) {
      // Replay decisions [applied, need), 32 at a time: the adds commute; the last lane of each
      // instance refreshes its terms once every add is in.
      bool abort = false;
      while ((int64_t)applied < need && !abort) {
        const uint32_t x = applied + (uint32_t)lane;
        const bool mine = (int64_t)x < need;
        unsigned long long jb = 0ull;
        if (mine) jb = wait_job(sync.jobs + x, err, sync.wait_ns);
        abort = __any_sync(0xffffffffu, mine && jb == 0ull);
        if (abort) break;
        const uint32_t j = mine ? job_pick(jb) : 0xFFFFFFFFu;
        const bool upd = mine && j < I;
        if (upd) {
          const uint32_t L = __ldg(&rows[x].L);
          const int64_t n = (int64_t)L - 16 * (int64_t)job_hit(jb);
          atomicAdd(&a.qr[j], 1);
          atomicAdd(reinterpret_cast<unsigned long long*>(&a.q[j]), (unsigned long long)n);
          atomicAdd(reinterpret_cast<unsigned long long*>(&a.S[j]), (unsigned long long)(int64_t)L);
        }
        const uint32_t nbatch = (int64_t)applied + 32 <= need ? 32u : (uint32_t)(need - (int64_t)applied);
        // the last 16 decisions of the batch take the ring slots (distinct within 16)
        if (mine && x + 16u >= applied + nbatch) s_jm[x & 15u] = j < I ? (int32_t)j : -1;
        const unsigned same = __match_any_sync(0xffffffffu, upd ? j : 0xFFFFFFFFu);
        __syncwarp();
        if (upd && (31 - __clz(same)) == lane) inst_refresh(a, m, j);
        __syncwarp();
        applied += nbatch;
      }
      c1 = clock64();
      if (lane == 0 && abort) s_abort = 1;
      if (lane < psk::kRowWords)
        reinterpret_cast<uint4*>(&s_row)[lane] = __ldg(reinterpret_cast<const uint4*>(rows + s) + lane);
    }
    __syncthreads();
    const long long c2 = clock64();
    if (t == 0) {
      cyc_job += (unsigned long long)(c1 - c0);
      cyc_ready += (unsigned long long)(c2 - c1);
    }
    if (s_abort) break;  // block-uniform
    const psk::RowConst rc = row_of(s_row);
    // raises from the picks of requests s - kLcpBack .. s - kSpecLag - 1 (older than the lag)
    constexpr int kNR = psk::kLcpBack - psk::kSpecLag;
    int32_t rj[kNR > 0 ? kNR : 1];
    uint32_t rl[kNR > 0 ? kNR : 1];
#pragma unroll
    for (int k2 = psk::kSpecLag; k2 < psk::kLcpBack; ++k2) {
      const int64_t t2 = (int64_t)s - 1 - k2;
      rj[k2 - psk::kSpecLag] = t2 >= 0 ? s_jm[(uint32_t)t2 & 15u] : -1;
      rl[k2 - psk::kSpecLag] = s_row.lcp[k2];
    }
    // every pair: hit, W, capacity guard, key in C
    PairKey pk[IPT];
    uint32_t hk[IPT];
    uint32_t wbest = 0xFFFFFFFFu;
#pragma unroll
    for (int k = 0; k < IPT; ++k) {
      const uint32_t i = t + (uint32_t)k * kPipeThreads;
      pk[k].inA = false;
      pk[k].key = psk::kNoKey;
      hk[k] = 0u;
      if (i < I) {
        const uint32_t h0 = hl[k];
        const uint32_t tp0 = tl[k];
        uint32_t h = h0;
#pragma unroll
        for (int q = 0; q < kNR; ++q)
          if (rj[q] == (int32_t)i && rl[q] > h) h = rl[q];
        hk[k] = h;
        pk[k] = pair_key_of(m, rc, a, i, h, h == h0 ? tp0 : psk::kNoTpfBits);
        if (pk[k].inA) wbest = min(wbest, psk::f2ord(pk[k].W));
      }
    }
    psk::RowSummary* out = sync.sums + (s % psk::kSumSlots);
    // per warp: W_min over A, its kWPerWarp smallest (W, instance), the next one as its bound
    {
      const uint32_t wm = __reduce_min_sync(0xffffffffu, wbest);
      if (lane == 0) s_wmin[warp] = wm;
      uint32_t taken = 0u;
#pragma unroll
      for (int rnd = 0; rnd <= psk::kWPerWarp; ++rnd) {
        unsigned long long mine = ~0ull;
        int mk = -1;
#pragma unroll
        for (int k = 0; k < IPT; ++k) {
          if (!pk[k].inA || ((taken >> k) & 1u)) continue;
          const unsigned long long w = ((unsigned long long)psk::f2ord(pk[k].W) << 32) | (t + (uint32_t)k * kPipeThreads);
          if (w < mine) {
            mine = w;
            mk = k;
          }
        }
        const unsigned long long best = warp_min_u64w(mine);
        if (mk >= 0 && mine == best) taken |= 1u << mk;
        if (rnd < psk::kWPerWarp) {
          if (lane == 0) out->w[warp * psk::kWPerWarp + rnd] = best;
        } else if (lane == 0) {
          s_wb[warp] = (uint32_t)(best >> 32);  // all ones when the warp has no more
        }
      }
    }
    __syncthreads();
    uint32_t wmin_o = 0xFFFFFFFFu;
#pragma unroll
    for (int w = 0; w < psk::kSumWarps; ++w) wmin_o = min(wmin_o, s_wmin[w]);
    const float wmin = psk::ord2f(wmin_o);
    // per warp: the kKeysPerWarp smallest (key, tie) of C, the next one as its bound
    {
      bool inC[IPT];
#pragma unroll
      for (int k = 0; k < IPT; ++k) inC[k] = pk[k].inA && psk::pair_in_c(rc, pk[k].W, wmin);
      uint32_t taken = 0u;
#pragma unroll
      for (int rnd = 0; rnd <= psk::kKeysPerWarp; ++rnd) {
        uint64_t bk = psk::kNoKey;
        uint32_t bt = 0xFFFFFFFFu, bh = 0u, bw = 0u;
        int mk = -1;
#pragma unroll
        for (int k = 0; k < IPT; ++k) {
          if (!inC[k] || ((taken >> k) & 1u)) continue;
          if (kt_less(pk[k].key, pk[k].tie, bk, bt)) {
            bk = pk[k].key;
            bt = pk[k].tie;
            bh = hk[k];
            bw = psk::f2ord(pk[k].W);
            mk = k;
          }
        }
        uint64_t wk;
        uint32_t wt, wh;
        psk::warp_pick_min(bk, bt, bh, &wk, &wt, &wh);
        const bool won = mk >= 0 && bk == wk && bt == wt;  // tie words are unique (instance in them)
        if (won) taken |= 1u << mk;
        const unsigned winm = __ballot_sync(0xffffffffu, won);
        const uint32_t ww = __shfl_sync(0xffffffffu, bw, winm ? __ffs(winm) - 1 : 0);
        if (rnd < psk::kKeysPerWarp) {
          if (lane == 0) {
            const int e = warp * psk::kKeysPerWarp + rnd;
            out->key[e] = wk;
            out->tie[e] = wt;
            out->word[e] = ww;
            out->hit[e] = wh;
          }
        } else if (lane == 0) {
          s_kb[warp] = wk;
          s_tb[warp] = wt;
        }
      }
    }
    __syncthreads();
    if (t == 0) {
      unsigned long long kb = psk::kNoKey;
      uint32_t tb = 0xFFFFFFFFu, wb = 0xFFFFFFFFu;
#pragma unroll
      for (int w = 0; w < psk::kSumWarps; ++w) {
        if (kt_less(s_kb[w], s_tb[w], kb, tb)) {
          kb = s_kb[w];
          tb = s_tb[w];
        }
        wb = min(wb, s_wb[w]);
      }
      out->key_bound = kb;
      out->tie_bound = tb;
      out->w_bound = wb;
      out->wmin = wmin_o;
      __threadfence();  // every warp's entries (written before the barrier) before the flag
      psk::st_release_u32(sync.sready + s, 1u);
      cyc_eval += (unsigned long long)(clock64() - c2);
    }
    __syncthreads();  // the next row reuses the reduction slots
  }
  if (t == 0 && sync.stats) {
    atomicAdd(sync.stats + psk::kGsSumJobWait, cyc_job);
    atomicAdd(sync.stats + psk::kGsSumReadyWait, cyc_ready);
    atomicAdd(sync.stats + psk::kGsSumEval, cyc_eval);
  }
}

// Deciding block: warp 0 decides, warp 1 (the feeder) stages rows in a shared-memory ring, warps 2, 3
// and 7 (the helpers A, B, C) prepare each step's inputs one step ahead, warp 5 hands decisions to
// them (and stores each pick's new state and writes the outputs); warps 4 and 6 return at once.  A
// warp's scheduler is warp id mod 4, so the spinning roles (deciding warp, feeder, warp 5) and the
// computing ones sit on different schedulers where they can.
//
// The decision of request s needs, besides row s's summary, the pairs on row s of the instances
// picked by decisions s - kSpecLag .. s - 1 under the current state: lane 0 the pick of s - 1, lane k
// the pick of s - 1 - k.  All but lane 0's depend only on decisions up to s - 2, and lane 0's is the
// winner of step s - 1 taking request s - 1.  So while step s - 1 is decided, the helpers compute for
// step s (their phase s - 1, started once decision s - 2 is published):
//   A[l]  summary entry l of row s - 1 as if it took request s - 1: its state after that, and its
//         pair on row s;
//   B[l]  the same for lane l's touched instance of step s - 1;
//   C[k]  the pick of s - 1 - k (k = 1 .. kSpecLag - 1) on row s under the state after s - 2.
// Step s then reads lane 0's pair from A, B (or, after a full pass or at the last request, from what
// the deciding warp computed itself, X) at the winner's index, and lane k's from C[k].  The deciding
// warp's own path is the W_min and key reductions of the corrected summary (whose entries it loads
// a step ahead) and one shared-memory publish; the helpers store each pick's new state into the
// instance arrays and write the decision outputs to global memory.
struct HelpSlot {
  PairKey a_pk[32];
  InstVals a_nv[32];
  uint32_t a_hit[32];
  int32_t a_qr[32];
  PairKey b_pk[psk::kSpecLag];
  InstVals b_nv[psk::kSpecLag];
  uint32_t b_hit[psk::kSpecLag];
  int32_t b_qr[psk::kSpecLag];
  PairKey c_pk[psk::kSpecLag];
  uint32_t c_hit[psk::kSpecLag];
  PairKey x_pk;
  InstVals x_nv;
  uint32_t x_hit;
  int32_t x_qr;
};
enum : uint32_t { kSrcA = 0, kSrcB = 1, kSrcX = 2 };
constexpr uint32_t kLogSlots = 64;  // decisions kept for the helpers (more than kLcpBack + 2)

// hit of instance c on row rw: its probed hit raised to the common prefix with each of the last
// kLcpBack requests that went to c (hist[k]: the pick of request s - 1 - k, s the step the history is
// taken at); `self` raises by lcp[0] too (c taking request s).  shift 0: rw is row s (lcp[k2] is with
// request s - 1 - k2 = hist[k2]); shift 1: rw is row s + 1 (lcp[k2] is with request s - k2 =
// hist[k2 - 1]).
__device__ __forceinline__ uint32_t raised_hit(const psk::RowPre& rw, const uint32_t* hr, uint32_t c, bool self, int shift,
                                               const int32_t (&hist)[psk::kLcpBack]) {
  uint32_t h = hr[c];
  if (self && rw.lcp[0] > h) h = rw.lcp[0];
#pragma unroll
  for (int k2 = 0; k2 < psk::kLcpBack; ++k2) {
    const int kk = k2 - shift;
    if (kk >= 0 && hist[kk < 0 ? 0 : kk] == (int32_t)c && rw.lcp[k2] > h) h = rw.lcp[k2];
  }
  return h;
}

// The as-if values of a decision's winner in a helper slot.
__device__ __forceinline__ const InstVals& slot_nv(const HelpSlot& hb, uint32_t src, uint32_t idx) {
  return src == kSrcA ? hb.a_nv[idx] : (src == kSrcB ? hb.b_nv[idx] : hb.x_nv);
}
__device__ __forceinline__ int32_t slot_qr(const HelpSlot& hb, uint32_t src, uint32_t idx) {
  return src == kSrcA ? hb.a_qr[idx] : (src == kSrcB ? hb.b_qr[idx] : hb.x_qr);
}
__device__ __forceinline__ uint32_t slot_hit(const HelpSlot& hb, uint32_t src, uint32_t idx) {
  return src == kSrcA ? hb.a_hit[idx] : (src == kSrcB ? hb.b_hit[idx] : hb.x_hit);
}

// Instance state v (of an instance with decode batch b, KV capacity M, slot limit Bmax and qr queued
// requests) after it takes a request of L tokens at hit h: inst_vals_after on given values.
__device__ __forceinline__ InstVals vals_after(const psk::DevModel& m, int32_t b, int64_t M, int32_t Bmax, int32_t qr0,
                                               const InstVals& v0, uint32_t L, uint32_t h, int32_t* qr_out) {
  const int32_t qr = qr0 + 1;
  InstVals v;
  v.q = v0.q + (int64_t)L - 16 * (int64_t)h;
  v.S = v0.S + (int64_t)L;
  const psk::InstTerms it = psk::inst_terms(m, b, qr, v.q, Bmax);
  v.dec0 = it.dec0;
  v.f = it.f;
  v.tq = it.tq;
  v.Bp = it.Bp;
  v.room = it.okB ? psk::kv_room(v.S, M) : -1;
  v.kd = psk::dcq_key0(b, qr);
  *qr_out = qr;
  return v;
}

__device__ void decide_spec(const psk::RowPre* __restrict__ rows, uint32_t R, uint32_t I, psk::StateSoA committed,
                            psk::StateSoA pending, const psk::DevModel& m, int32_t* assign, uint8_t* __restrict__ path,
                            uint32_t* __restrict__ hit_chosen, uint32_t* err, const psk::GreedySync& sync,
                            unsigned long long* smem_raw) {
  const int wid = (int)(threadIdx.x >> 5);
  if (wid == 4 || wid == 6) return;
  const uint32_t Ip = sync.ring_stride;
  const InstSmem a = inst_smem(smem_raw, Ip);
  uint32_t* s_hitr = reinterpret_cast<uint32_t*>(a.Bmax + Ip);  // [kFeedRing][Ip] probed hits
  uint32_t* s_tpfr = s_hitr + kFeedRing * Ip;                   // [kFeedRing][Ip] T_pf at them (bits)
  __shared__ psk::RowSummary s_sum[kFeedRing];
  __shared__ psk::RowPre s_rowc[kFeedRing];
  __shared__ HelpSlot s_help[2];               // helper phase p writes s_help[p & 1]
  __shared__ int32_t s_logpick[kLogSlots];     // decision x: its pick (-1 rejected) ...
  __shared__ uint32_t s_logsrc[kLogSlots];     // ... where its as-if values are (kSrc*) and at which index
  __shared__ uint32_t s_logidx[kLogSlots];
  __shared__ uint32_t s_loghit[kLogSlots];     // ... its hit and path (the decision outputs)
  __shared__ uint32_t s_logpath[kLogSlots];
  __shared__ uint32_t s_fed;       // rows [0, s_fed) are staged (release / acquire)
  __shared__ uint32_t s_dec;       // decisions [0, s_dec) are published (their rows are consumed)
  __shared__ uint32_t s_stored;    // the state after decisions [0, s_stored) is in the instance arrays
  __shared__ uint32_t s_ph[3];     // helper w (A, B, C) finished phases [0, s_ph[w])
  __shared__ int s_hgo[2];         // helper phase p goes ahead (s_hgo[p & 1]), set before its barrier
  __shared__ volatile int s_stop;  // a role gave up (a bounded wait ran out)
  const uint32_t t = threadIdx.x;
  const int lane = (int)(t & 31u), warp = (int)(t >> 5);
  const unsigned full = 0xffffffffu;
  if (t < 64)
    for (uint32_t i = t; i < I; i += 64) inst_load(a, committed, m, i);
  if (t == 0) {
    s_fed = 0u;
    s_dec = 0u;
    s_stored = 0u;
    s_ph[0] = 0u;
    s_ph[1] = 0u;
    s_ph[2] = 0u;
    s_stop = 0;
  }
  asm volatile("bar.sync 1, 192;" ::: "memory");  // warps 0, 1, 2, 3, 5, 7

  if (warp == 1) {
    // ---- feeder ---------------------------------------------------------------------------------
    // Row x's slot held row x - kFeedRing, which the deciding warp reads up to its decision
    // x - kFeedRing and the helpers up to their phase x - kFeedRing.
    unsigned long long cyc_slot = 0, cyc_sum = 0;
    for (uint32_t x = 0; x < R; ++x) {
      const uint32_t slot = x % kFeedRing;
      bool ok = true;
      if (lane == 0) {
        const long long c0 = clock64();
        if (x >= kFeedRing) {
          const uint32_t want = x - kFeedRing + 1;
          ok = wait_smem_at_least(&s_dec, want, &s_stop, err, sync.wait_ns) &&
               wait_smem_at_least(&s_ph[0], want, &s_stop, err, sync.wait_ns) &&
               wait_smem_at_least(&s_ph[1], want, &s_stop, err, sync.wait_ns) &&
               wait_smem_at_least(&s_ph[2], want, &s_stop, err, sync.wait_ns);
        }
        const long long c1 = clock64();
        if (ok) ok = wait_flag(sync.sready + x, err, sync.wait_ns);
        cyc_slot += (unsigned long long)(c1 - c0);
        cyc_sum += (unsigned long long)(clock64() - c1);
        if (!ok) s_stop = 1;
      }
      ok = __shfl_sync(full, ok ? 1 : 0, 0) != 0;
      __syncwarp();
      if (!ok) break;  // warp-uniform
      const uint4* src_sum = reinterpret_cast<const uint4*>(sync.sums + (x % psk::kSumSlots));
      uint4* dst_sum = reinterpret_cast<uint4*>(&s_sum[slot]);
      for (uint32_t w = (uint32_t)lane; w < sizeof(psk::RowSummary) / 16; w += 32) psk::cp_async16(dst_sum + w, src_sum + w);
      if (lane < psk::kRowWords)
        psk::cp_async16(reinterpret_cast<uint4*>(&s_rowc[slot]) + lane, reinterpret_cast<const uint4*>(rows + x) + lane);
      const uint4* src_h = reinterpret_cast<const uint4*>(sync.hitring + (uint64_t)(x % psk::kHitSlots) * Ip);
      const uint4* src_t = reinterpret_cast<const uint4*>(sync.tpfring + (uint64_t)(x % psk::kHitSlots) * Ip);
      uint4* dst_h = reinterpret_cast<uint4*>(s_hitr + slot * Ip);
      uint4* dst_t = reinterpret_cast<uint4*>(s_tpfr + slot * Ip);
      for (uint32_t w = (uint32_t)lane; w < Ip / 4; w += 32) {
        psk::cp_async16(dst_h + w, src_h + w);
        psk::cp_async16(dst_t + w, src_t + w);
      }
      psk::cp_async_commit();
      psk::cp_async_wait_all();
      __syncwarp();
      if (lane == 0) psk::st_release_cta_shared_u32(&s_fed, x + 1);
    }
    if (lane == 0 && sync.stats) {
      atomicAdd(sync.stats + psk::kGsFeedSlotWait, cyc_slot);
      atomicAdd(sync.stats + psk::kGsFeedSumWait, cyc_sum);
    }
    return;
  }

  if (warp >= 2) {
    // ---- helpers ----------------------------------------------------------------------------------
    // Phase p (p = 0 .. R): once decision p - 1 is published, warp 5 stores its pick's new state and
    // writes its outputs, and for p < R - 1 the helpers compute A (warp 2), B (warp 3) and C (warp 7)
    // for step p + 1 into s_help[p & 1].  Lanes whose instance is the pick of p - 1 take its state from
    // the winner's as-if values, so nothing waits for the store: the others' instances were not
    // picked at p - 1.
    const int role = warp == 2 ? 0 : (warp == 3 ? 1 : (warp == 7 ? 2 : 3));  // 3: warp 5
    for (uint32_t p = 0; p <= R; ++p) {
      if (role == 3 && lane == 0) {
        bool ok = wait_smem_at_least(&s_dec, p, &s_stop, err, sync.wait_ns);
        if (ok && p < R) ok = wait_smem_at_least(&s_fed, p + 2 < R ? p + 2 : R, &s_stop, err, sync.wait_ns);
        if (!ok) s_stop = 1;
        s_hgo[p & 1u] = ok ? 1 : 0;
      }
      asm volatile("bar.sync 2, 128;" ::: "memory");  // warps 2, 3, 5, 7
      if (!s_hgo[p & 1u]) break;  // uniform across the helper warps
      const HelpSlot& hp = s_help[(p - 1) & 1u];  // phase p - 1's slot (p >= 1)
      const uint32_t xp = (p - 1) % kLogSlots;     // decision p - 1 in the log (p >= 1)
      int32_t j0 = -1;                              // the pick of p - 1
      uint32_t src0 = kSrcX, idx0 = 0u;
      if (p >= 1) {
        j0 = s_logpick[xp];
        src0 = s_logsrc[xp];
        idx0 = s_logidx[xp];
      }
      if (role == 3) {
        if (lane == 0) {
          if (j0 >= 0) inst_store(a, (uint32_t)j0, slot_qr(hp, src0, idx0), slot_nv(hp, src0, idx0));
          psk::st_release_cta_shared_u32(&s_stored, p);
        } else if (lane == 1 && p >= 1) {
          assign[p - 1] = j0;
          path[p - 1] = (uint8_t)s_logpath[xp];
          hit_chosen[p - 1] = s_loghit[xp];
        }
        continue;
      }
      if (p == R) break;
      if (p + 1 >= R) {  // no row R: nothing to compute
        __syncwarp();
        if (lane == 0) psk::st_release_cta_shared_u32(&s_ph[role], p + 1);
        continue;
      }
      int32_t hist[psk::kLcpBack];
#pragma unroll
      for (int k = 0; k < psk::kLcpBack; ++k)
        hist[k] = (int64_t)p - 1 - k >= 0 ? s_logpick[(p - 1 - k) % kLogSlots] : -1;
      const uint32_t slot = p % kFeedRing, slot1 = (p + 1) % kFeedRing;
      const psk::RowPre& row = s_rowc[slot];
      const psk::RowPre& row1 = s_rowc[slot1];
      const psk::RowConst rc1 = row_of(row1);
      const uint32_t* hrow1 = s_hitr + slot1 * Ip;
      const uint32_t* trow1 = s_tpfr + slot1 * Ip;
      HelpSlot& out = s_help[p & 1u];
      // instance c (state v0, qr0) taking request p at hit h: its state after, and its pair on row p + 1
      auto as_if = [&](uint32_t c, const InstVals& v0, int32_t qr0, uint32_t h, PairKey* pk, InstVals* nv,
                       uint32_t* hit, int32_t* qr) {
        *nv = vals_after(m, a.b[c], a.M[c], a.Bmax[c], qr0, v0, row.L, h, qr);
        *hit = raised_hit(row1, hrow1, c, true, 1, hist);
        *pk = pair_key_v(m, rc1, *nv, c, *hit, *hit == hrow1[c] ? trow1[c] : psk::kNoTpfBits);
      };
      if (role == 0) {
        // A: summary entry `lane` of row p, when no decision of the last kSpecLag picked it (its state
        // is then the one in the instance arrays)
        const psk::RowSummary& sm = s_sum[slot];
        const uint64_t ek = sm.key[lane];
        const uint32_t e = sm.tie[lane] & psk::kTieInstMask;
        bool touched = false;
#pragma unroll
        for (int k = 0; k < psk::kSpecLag; ++k) touched |= hist[k] == (int32_t)e;
        if (ek != psk::kNoKey && !touched) {
          PairKey pk;
          InstVals nv;
          uint32_t hit;
          int32_t qr;
          as_if(e, inst_vals(a, e), a.qr[e], sm.hit[lane], &pk, &nv, &hit, &qr);
          out.a_pk[lane] = pk;
          out.a_nv[lane] = nv;
          out.a_hit[lane] = hit;
          out.a_qr[lane] = qr;
        }
      } else if (role == 1) {
        // B: lane's touched instance of step p (the pick of p - 1 - lane) as if it took request p, at
        // its hit on row p (from phase p - 1)
        const int32_t u = lane < psk::kSpecLag && (int64_t)p - 1 - lane >= 0 ? s_logpick[(p - 1 - lane) % kLogSlots] : -1;
        if (u >= 0) {
          PairKey pk;
          InstVals nv;
          uint32_t hit;
          int32_t qr;
          // lane 0's instance is the pick of p - 1: its state is the winner's as-if values (one call for
          // every lane, so the lanes do not diverge)
          const InstVals v0 = lane == 0 ? slot_nv(hp, src0, idx0) : inst_vals(a, (uint32_t)u);
          const int32_t qr0 = lane == 0 ? slot_qr(hp, src0, idx0) : a.qr[u];
          const uint32_t h0 = lane == 0 ? slot_hit(hp, src0, idx0) : hp.c_hit[lane];
          as_if((uint32_t)u, v0, qr0, h0, &pk, &nv, &hit, &qr);
          out.b_pk[lane] = pk;
          out.b_nv[lane] = nv;
          out.b_hit[lane] = hit;
          out.b_qr[lane] = qr;
        }
      } else {
        // C: the pick of p - k (k = lane, 1 .. kSpecLag - 1) on row p + 1, current state
        const int k = lane;
        const int32_t u = k >= 1 && k < psk::kSpecLag && (int64_t)p - k >= 0 ? s_logpick[(p - k) % kLogSlots] : -1;
        if (u >= 0) {
          const uint32_t h = raised_hit(row1, hrow1, (uint32_t)u, false, 1, hist);
          const uint32_t tb = h == hrow1[u] ? trow1[u] : psk::kNoTpfBits;
          out.c_pk[k] = pair_key_v(m, rc1, k == 1 ? slot_nv(hp, src0, idx0) : inst_vals(a, (uint32_t)u), (uint32_t)u, h, tb);
          out.c_hit[k] = h;
        }
      }
      __syncwarp();
      if (lane == 0) psk::st_release_cta_shared_u32(&s_ph[role], p + 1);
    }
    return;
  }

  // ---- deciding warp --------------------------------------------------------------------------------
  //   pk     lane k < kLcpBack: the pick of request s - 1 - k (-1: none or rejected)
  //   hist   the same picks in every lane
  //   cor    lane k < kSpecLag: that instance's pair on row s under the current state, chit its hit
  //   e*, w* this lane's summary entries of row s, loaded a step ahead
  int32_t pk = -1;
  int32_t hist[psk::kLcpBack];
#pragma unroll
  for (int k = 0; k < psk::kLcpBack; ++k) hist[k] = -1;
  uint32_t w_src = kSrcA, w_idx = 0;  // where the previous winner's as-if values are
  unsigned long long n_fast = 0, n_full = 0, cyc_wait = 0;
  const long long cyc_start = clock64();
  uint64_t ek = psk::kNoKey, wv = ~0ull, kbound = psk::kNoKey;
  uint32_t et = 0u, ew = 0u, eh = 0u, wbound = 0u, wsum = 0u, tbound = 0u;
  psk::RowConst rc{};
  auto load_row = [&](uint32_t x) {
    const psk::RowSummary& sm = s_sum[x % kFeedRing];
    ek = sm.key[lane];
    et = sm.tie[lane];
    ew = sm.word[lane];
    eh = sm.hit[lane];
    wv = lane < psk::kSumWarps * psk::kWPerWarp ? sm.w[lane] : ~0ull;
    wbound = sm.w_bound;
    wsum = sm.wmin;
    kbound = sm.key_bound;
    tbound = sm.tie_bound;
    rc = row_of(s_rowc[x % kFeedRing]);
  };
  for (uint32_t s = 0; s < R; ++s) {
    const uint32_t slot = s % kFeedRing;
    const bool has_next = s + 1 < R;
    bool ok = true;
    if (lane == 0) {
      const long long c0 = clock64();
      ok = wait_smem_at_least(&s_fed, has_next ? s + 2 : s + 1, &s_stop, err, sync.wait_ns);
      if (ok && s >= 1)
        ok = wait_smem_at_least(&s_ph[0], s, &s_stop, err, sync.wait_ns) &&
             wait_smem_at_least(&s_ph[1], s, &s_stop, err, sync.wait_ns) &&
             wait_smem_at_least(&s_ph[2], s, &s_stop, err, sync.wait_ns);
      cyc_wait += (unsigned long long)(clock64() - c0);
      if (!ok) s_stop = 1;
    }
    ok = __shfl_sync(full, ok ? 1 : 0, 0) != 0;
    __syncwarp();
    if (!ok) break;  // warp-uniform
    if (s == 0) load_row(0);
    PairKey cor;
    cor.W = 0.0f;
    cor.key = psk::kNoKey;
    cor.tie = 0xFFFFFFFFu;
    cor.inA = false;
    uint32_t chit = 0u;
    if (s >= 1 && lane < psk::kSpecLag && pk >= 0) {
      const HelpSlot& hb = s_help[(s - 1) & 1u];
      if (lane == 0) {
        cor = w_src == kSrcA ? hb.a_pk[w_idx] : (w_src == kSrcB ? hb.b_pk[w_idx] : hb.x_pk);
        chit = slot_hit(hb, w_src, w_idx);
      } else {
        cor = hb.c_pk[lane];
        chit = hb.c_hit[lane];
      }
    }
    auto touched = [&](uint32_t i) {
      bool r = false;
#pragma unroll
      for (int k = 0; k < psk::kSpecLag; ++k) r |= hist[k] == (int32_t)i;
      return r;
    };
    // the touched instances, one lane each (the latest occurrence)
    const int32_t tk = lane < psk::kSpecLag ? pk : -1;
    const unsigned same = __match_any_sync(full, tk);
    const bool corr = tk >= 0 && (__ffs(same) - 1) == lane;
    // W_min of the current state
    const bool w_untouched = wv != ~0ull && !touched((uint32_t)wv);
    const uint32_t mu = __reduce_min_sync(full, w_untouched ? (uint32_t)(wv >> 32) : 0xFFFFFFFFu);
    const uint32_t mt = __reduce_min_sync(full, (corr && cor.inA) ? psk::f2ord(cor.W) : 0xFFFFFFFFu);
    uint32_t wmin_o = min(mu, mt);
    bool anyA = wmin_o != 0xFFFFFFFFu;
    bool fast = wbound == 0xFFFFFFFFu || mu <= wbound;
    if (fast && anyA && rc.Z > 0.0f && wmin_o > wsum) fast = false;
    // this lane's candidate: its summary entry or its touched instance, whichever is smaller
    uint64_t bk = psk::kNoKey;
    uint32_t bt = 0xFFFFFFFFu, bh = 0u, bsrc = kSrcA;
    if (fast && anyA) {
      const float wmin = psk::ord2f(wmin_o);
      if (ek != psk::kNoKey && !touched(et & psk::kTieInstMask) && psk::pair_in_c(rc, psk::ord2f(ew), wmin)) {
        bk = ek;
        bt = et;
        bh = eh;
      }
      if (corr && cor.inA && psk::pair_in_c(rc, cor.W, wmin) && kt_less(cor.key, cor.tie, bk, bt)) {
        bk = cor.key;
        bt = cor.tie;
        bh = chit;
        bsrc = kSrcB;
      }
    }
    uint64_t K = psk::kNoKey;
    uint32_t T = 0xFFFFFFFFu, H = 0u;
    if (fast && anyA) {
      psk::warp_pick_min(bk, bt, bh, &K, &T, &H);
      fast = K != psk::kNoKey && (kbound == psk::kNoKey || kt_less(K, T, kbound, tbound));
    }
    const bool won = fast && bk != psk::kNoKey && bk == K && bt == T;  // one lane at most (tie words are unique)
    const psk::RowPre& row = s_rowc[slot];
    const uint32_t* hrow = s_hitr + slot * Ip;
    const uint32_t* trow = s_tpfr + slot * Ip;
    bool stored = false;  // the state after decision s - 1 is known to be in the instance arrays
    if (fast) {
      ++n_fast;
    } else {
      // full pass over the row on the current state (which needs the previous pick's state stored)
      ++n_full;
      bool ok2 = true;
      if (lane == 0) {
        ok2 = wait_smem_at_least(&s_stored, s, &s_stop, err, sync.wait_ns);
        if (!ok2) s_stop = 1;
      }
      ok2 = __shfl_sync(full, ok2 ? 1 : 0, 0) != 0;
      __syncwarp();
      if (!ok2) break;  // warp-uniform
      stored = true;
      uint32_t wo = 0xFFFFFFFFu;
      for (uint32_t i = (uint32_t)lane; i < I; i += 32) {
        if ((int32_t)rc.L <= a.room[i]) {
          const uint32_t h = raised_hit(row, hrow, i, false, 0, hist);
          const float tpf = (h == hrow[i] && trow[i] != psk::kNoTpfBits) ? __uint_as_float(trow[i]) : psk::t_pf32(m, rc.L, h);
          wo = min(wo, psk::f2ord(__fsub_rn(tpf, rc.t_cached)));
        }
      }
      wmin_o = __reduce_min_sync(full, wo);
      anyA = wmin_o != 0xFFFFFFFFu;
      const float wmin = psk::ord2f(wmin_o);
      uint64_t fk = psk::kNoKey;
      uint32_t ft = 0xFFFFFFFFu, fh = 0u;
      if (anyA) {
        for (uint32_t i = (uint32_t)lane; i < I; i += 32) {
          const uint32_t h = raised_hit(row, hrow, i, false, 0, hist);
          const PairKey p = pair_key_of(m, rc, a, i, h, h == hrow[i] ? trow[i] : psk::kNoTpfBits);
          if (p.inA && psk::pair_in_c(rc, p.W, wmin) && kt_less(p.key, p.tie, fk, ft)) {
            fk = p.key;
            ft = p.tie;
            fh = h;
          }
        }
      }
      psk::warp_pick_min(fk, ft, fh, &K, &T, &H);
    }
    const bool pick = anyA && K != psk::kNoKey;
    const uint32_t j = T & psk::kTieInstMask;
    if (!pick) H = 0u;
    // where the pick's as-if values (its state after this decision, its pair on row s + 1) are
    uint32_t src = kSrcX, idx = 0u;
    const unsigned wm = __ballot_sync(full, won);
    if (wm && has_next) {
      const int wl = __ffs(wm) - 1;
      src = __shfl_sync(full, bsrc, wl);
      idx = (uint32_t)wl;
    } else if (pick) {
      // a full pass picked it (the helpers prepared no such candidate), or the last request (there is
      // no next row): its values are computed here, on the stored state
      bool ok3 = true;
      if (lane == 0) {
        if (!stored) ok3 = wait_smem_at_least(&s_stored, s, &s_stop, err, sync.wait_ns);
        if (ok3) {
          HelpSlot& xb = s_help[s & 1u];
          int32_t qr2;
          const InstVals v2 = inst_vals_after(a, m, j, rc.L, H, &qr2);
          xb.x_nv = v2;
          xb.x_qr = qr2;
          if (has_next) {
            const uint32_t slot1 = (s + 1) % kFeedRing;
            const psk::RowPre& row1 = s_rowc[slot1];
            const uint32_t* hrow1 = s_hitr + slot1 * Ip;
            const uint32_t* trow1 = s_tpfr + slot1 * Ip;
            const uint32_t h1 = raised_hit(row1, hrow1, j, true, 1, hist);
            xb.x_pk = pair_key_v(m, row_of(row1), v2, j, h1, h1 == hrow1[j] ? trow1[j] : psk::kNoTpfBits);
            xb.x_hit = h1;
          }
        } else {
          s_stop = 1;
        }
      }
      __syncwarp();
    }
    if (lane == 0) {
      const uint32_t x = s % kLogSlots;
      s_logpick[x] = pick ? (int32_t)j : -1;
      s_logsrc[x] = src;
      s_logidx[x] = idx;
      s_loghit[x] = H;
      s_logpath[x] = pick ? (uint32_t)(K >> 62) : 2u;
      psk::st_release_cta_shared_u32(&s_dec, s + 1);
      psk::st_relaxed_u64(sync.jobs + s, kJobValid | ((unsigned long long)H << 32) | (pick ? j : 0xFFFFFFFFu));
    }
    const int32_t pj = pick ? (int32_t)j : -1;
    pk = __shfl_up_sync(full, pk, 1);
    if (lane == 0) pk = pj;
#pragma unroll
    for (int k = psk::kLcpBack - 1; k > 0; --k) hist[k] = hist[k - 1];
    hist[0] = pj;
    w_src = src;
    w_idx = idx;
    if (has_next) load_row(s + 1);  // staged: s_fed >= s + 2 was waited for
  }
  if (lane == 0 && sync.stats) {
    atomicAdd(sync.stats + psk::kGsFast, n_fast);
    atomicAdd(sync.stats + psk::kGsFull, n_full);
    atomicAdd(sync.stats + psk::kGsDecideWait, cyc_wait);
    atomicAdd(sync.stats + psk::kGsDecideTotal, (unsigned long long)(clock64() - cyc_start));
  }
  // the pending state: every decision's state stored by the helpers (their phase R)
  bool ok = true;
  if (lane == 0) ok = !s_stop && wait_smem_at_least(&s_stored, R, &s_stop, err, sync.wait_ns);
  ok = __shfl_sync(full, ok ? 1 : 0, 0) != 0;
  if (!ok) return;
  for (uint32_t i = (uint32_t)lane; i < I; i += 32) {
    pending.b[i] = a.b[i];
    pending.qr[i] = a.qr[i];
    pending.q[i] = a.q[i];
    pending.S[i] = a.S[i];
    pending.M[i] = a.M[i];
    pending.Bmax[i] = a.Bmax[i];
  }
}

template <int IPT>
__global__ void __launch_bounds__(kPipeThreads, 1)
greedy_pipe_kernel(const psk::RowPre* __restrict__ rows, const uint64_t* __restrict__ hash, uint32_t R, uint32_t I,
                   const uint32_t* __restrict__ hit0, const float* __restrict__ tpf0, psk::StateSoA committed,
                   psk::StateSoA pending, psk::DevModel m, psk::DeltaSlot* delta, uint64_t nslots, int32_t* assign,
                   uint8_t* __restrict__ path, uint32_t* __restrict__ hit_chosen, uint32_t* err, psk::GreedySync sync) {
  extern __shared__ unsigned long long smem_raw[];
  if (blockIdx.x == 0) {
    decide_spec(rows, R, I, committed, pending, m, assign, path, hit_chosen, err, sync, smem_raw);
  } else if (blockIdx.x <= kInsertBlocks) {
    insert_blocks(rows, hash, R, delta, nslots, err, sync);
  } else if (blockIdx.x <= kInsertBlocks + kProbeBlocks) {
    probe_rows<IPT>(rows, hash, R, I, hit0, tpf0, delta, nslots, err, sync, smem_raw);
  } else {
    summary_rows<IPT>(rows, R, I, committed, m, err, sync, blockIdx.x - 1 - kInsertBlocks - kProbeBlocks, smem_raw);
  }
}

size_t greedy_pipe_smem(uint32_t I, uint32_t Ip) {
  // deciding block: instance state, the hit and T_pf rows of kFeedRing rows; summary blocks: the
  // instance state; probe blocks: three u32 arrays per instance
  const size_t decide = (size_t)Ip * (kInstSmemBytes + 2 * kFeedRing * sizeof(uint32_t));
  const size_t probe = (size_t)I * 3 * sizeof(uint32_t);
  return decide > probe ? decide : probe;
}

template <int IPT>
cudaError_t greedy_pipe_launch(const psk::RowPre* rows, const psk::WindowDev& w, uint32_t I, const uint32_t* hit0,
                               const float* tpf0, psk::StateSoA committed, psk::StateSoA pending, const psk::DevModel& m,
                               psk::DeltaSlot* delta, uint64_t nslots, int32_t* assign, uint8_t* path,
                               uint32_t* hit_chosen, uint32_t* err, const psk::GreedySync& sync, cudaStream_t s) {
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
  return cudaLaunchCooperativeKernel((const void*)greedy_pipe_kernel<IPT>,
                                     dim3(1 + kInsertBlocks + kProbeBlocks + kSummaryBlocks), dim3(kPipeThreads), args,
                                     smem, s);
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
  if (e == cudaSuccess) e = cudaMemsetAsync(sync.sready, 0, (size_t)w.R * sizeof(uint32_t), s);
  if (e == cudaSuccess) e = cudaMemsetAsync(sync.jobs, 0, (size_t)w.R * sizeof(unsigned long long), s);
  if (e == cudaSuccess && sync.stats) e = cudaMemsetAsync(sync.stats, 0, psk::kGreedyStats * sizeof(unsigned long long), s);
  if (e != cudaSuccess) return e;
  // every block has 256 threads; probe and summary threads hold IPT = ceil(I / 256) instances each
  const uint32_t ipt = (I + kPipeThreads - 1) / kPipeThreads;
#define PS_GREEDY_P(IPT)                                                                                      \
  return greedy_pipe_launch<IPT>(rows, w, I, hit0, tpf0, committed, pending, m, delta, delta_nslots, assign, path, \
                                 hit_chosen, err, sync, s)
  if (ipt <= 1) PS_GREEDY_P(1);
  if (ipt <= 2) PS_GREEDY_P(2);
  if (ipt <= 4) PS_GREEDY_P(4);
  if (ipt <= 8) PS_GREEDY_P(8);
#undef PS_GREEDY_P
  return cudaErrorInvalidValue;
}

// The delta table only holds one window's blocks: clear it whole after each window.
cudaError_t launch_delta_clear(psk::DeltaSlot* delta, uint64_t nslots, cudaStream_t s) {
  return cudaMemsetAsync(delta, 0, nslots * sizeof(psk::DeltaSlot), s);
}

}  // namespace pskl
