// Table maintenance and between-window kernels: bulk insertion of cached chains, commit of a
// scheduled window, engine progress of a streaming window, leaf-first LRU eviction, the
// prefix-closure check and the device-side window layout check.
#include "ps_internal.cuh"

namespace {

// Bulk insert: one warp per instance, the instance's only writer.  The warp scans the chain list
// 32 entries at a time for its own chains and inserts their blocks in order (balanced two-choice
// placement needs the current bucket fill, so each table is written sequentially; different
// instances proceed in parallel).  Block 0 of chain c continues parent[c], block k continues k-1.
__global__ void insert_chains_kernel(uint64_t* slots, uint64_t* ovf, const psk::TableDesc* __restrict__ tdesc,
                                     uint32_t I, unsigned long long* count, uint64_t nchains,
                                     const uint32_t* __restrict__ inst, const uint64_t* __restrict__ off,
                                     const uint64_t* __restrict__ hash, const uint64_t* __restrict__ parent,
                                     psk::LruMeta meta, uint32_t last_use, uint32_t* err) {
  const int lane = threadIdx.x & 31;
  const uint32_t warps_total = (gridDim.x * blockDim.x) >> 5;
  for (uint32_t i = (blockIdx.x * blockDim.x + threadIdx.x) >> 5; i < I; i += warps_total) {
    const psk::TableDesc d = tdesc[i];
    unsigned long long added = 0;
    bool full = false, reserved = false;
    for (uint64_t c0 = 0; c0 < nchains; c0 += 32) {
      const uint64_t c = c0 + lane;
      unsigned mine = __ballot_sync(0xffffffffu, c < nchains && __ldg(inst + c) == i);
      while (mine) {
        const int l = __ffs(mine) - 1;
        mine &= mine - 1;
        const uint64_t a = __ldg(off + c0 + l), b = __ldg(off + c0 + l + 1);
        uint64_t prev_key = __ldg(parent + c0 + l), prev_slot = ~0ull;
        for (uint64_t k = a; k < b && !full; ++k) {
          const uint64_t key = __ldg(hash + k);
          if (key == psk::kEmpty || key == psk::kTomb) {
            reserved = true;
            prev_key = key;
            prev_slot = ~0ull;
            continue;
          }
          bool ins = false;
          const uint64_t slot = psk::warp_insert(slots, ovf, d, key, &ins, meta, prev_key, last_use, prev_slot);
          if (slot == ~0ull) full = true;
          if (ins) ++added;
          prev_key = key;
          prev_slot = slot;
        }
      }
    }
    if (lane == 0) {
      count[i] += added;
      if (full) atomicOr(err, psk::kErrTableFull);
      if (reserved) atomicOr(err, psk::kErrReservedHash);
    }
  }
}

// Instance ids must be valid before the per-instance scan (a chain with a bad id is never seen).
__global__ void check_instances_kernel(uint32_t I, uint64_t nchains, const uint32_t* __restrict__ inst,
                                       uint32_t* err) {
  for (uint64_t c = blockIdx.x * (uint64_t)blockDim.x + threadIdx.x; c < nchains; c += (uint64_t)gridDim.x * blockDim.x)
    if (inst[c] >= I) atomicOr(err, psk::kErrBadInstance);
}

// Commit of a scheduled window, in four passes over every admitted request's blocks (within a window
// each (block, instance) pair is inserted at most once: a request inserts chain[h, nb) on its pick
// with h the exact first miss there, so none of those blocks is cached on that instance yet, neither
// by the committed caches nor by an earlier request):
//   stamp   the cached prefix chain[0, h) gets last_use (every stamp writes the same value, so
//           their order does not matter);
//   insert  the uncached blocks chain[h, nb) are cached, stamped, with 0 children and their parent
//           link pending;
//   link    each new block records its parent's slot and the parent gains a child;
//   queue   with request tracking, each instance appends its admitted requests to its FIFO queue
//           in arrival order (one warp per instance).
// The first three run over one flat index space of (request, block) items, so a long chain is
// spread over the whole grid: a prefix pass gives each admitted request its first item, and an item
// finds its request by binary search.

// Exclusive prefix sums over the window's requests of the items of the stamp pass (h) and of the
// insert and link passes (nb - h); rejected requests have none.  One block; pre_s and pre_i hold
// R + 1 entries each.
__global__ void __launch_bounds__(1024)
commit_prefix_kernel(psk::WindowDev w, const int32_t* __restrict__ assign, const uint32_t* __restrict__ hit_chosen,
                     unsigned long long* pre_s, unsigned long long* pre_i) {
  __shared__ unsigned long long s_ws[32], s_wi[32];
  __shared__ unsigned long long s_carry_s, s_carry_i;
  const uint32_t t = threadIdx.x, lane = t & 31u, warp = t >> 5;
  if (t == 0) {
    s_carry_s = 0ull;
    s_carry_i = 0ull;
  }
  __syncthreads();
  for (uint32_t r0 = 0; r0 < w.R; r0 += blockDim.x) {
    const uint32_t r = r0 + t;
    unsigned long long cs = 0ull, ci = 0ull;
    if (r < w.R && assign[r] >= 0) {
      const uint64_t h = hit_chosen[r];
      const uint64_t nb = w.off[r + 1] - w.off[r];
      cs = h;
      ci = nb > h ? nb - h : 0ull;
    }
    unsigned long long xs = cs, xi = ci;  // inclusive warp scans
#pragma unroll
    for (int d = 1; d < 32; d <<= 1) {
      const unsigned long long ys = __shfl_up_sync(0xffffffffu, xs, d), yi = __shfl_up_sync(0xffffffffu, xi, d);
      if ((int)lane >= d) {
        xs += ys;
        xi += yi;
      }
    }
    if (lane == 31u) {
      s_ws[warp] = xs;
      s_wi[warp] = xi;
    }
    __syncthreads();
    if (warp == 0) {
      const uint32_t nw = blockDim.x >> 5;
      unsigned long long vs = lane < nw ? s_ws[lane] : 0ull, vi = lane < nw ? s_wi[lane] : 0ull;
#pragma unroll
      for (int d = 1; d < 32; d <<= 1) {
        const unsigned long long ys = __shfl_up_sync(0xffffffffu, vs, d), yi = __shfl_up_sync(0xffffffffu, vi, d);
        if ((int)lane >= d) {
          vs += ys;
          vi += yi;
        }
      }
      // exclusive warp offsets from the inclusive ones
      const unsigned long long es = __shfl_up_sync(0xffffffffu, vs, 1), ei = __shfl_up_sync(0xffffffffu, vi, 1);
      if (lane < nw) {
        s_ws[lane] = lane == 0 ? 0ull : es;
        s_wi[lane] = lane == 0 ? 0ull : ei;
      }
    }
    __syncthreads();
    if (r < w.R) {
      pre_s[r] = s_carry_s + s_ws[warp] + xs - cs;
      pre_i[r] = s_carry_i + s_wi[warp] + xi - ci;
    }
    __syncthreads();
    if (t == blockDim.x - 1u) {  // the chunk's total carries into the next chunk
      s_carry_s += s_ws[warp] + xs;
      s_carry_i += s_wi[warp] + xi;
    }
    __syncthreads();
  }
  if (t == 0) {
    pre_s[w.R] = s_carry_s;
    pre_i[w.R] = s_carry_i;
  }
}

// The request of flat item x: the last r with pre[r] <= x (pre ascending, pre[0] = 0, x < pre[R]).
__device__ __forceinline__ uint32_t item_request(const unsigned long long* __restrict__ pre, uint32_t R,
                                                 unsigned long long x) {
  uint32_t lo = 0, hi = R;  // pre[lo] <= x < pre[hi]
  while (hi - lo > 1u) {
    const uint32_t mid = (lo + hi) >> 1;
    if (__ldg(pre + mid) <= x) lo = mid;
    else hi = mid;
  }
  return lo;
}

__global__ void commit_stamp_kernel(const uint64_t* slots, const uint64_t* ovf, const psk::TableDesc* __restrict__ tdesc,
                                    psk::WindowDev w, const int32_t* __restrict__ assign,
                                    const unsigned long long* __restrict__ pre_s, psk::LruMeta meta, uint32_t last_use) {
  const unsigned long long total = pre_s[w.R];
  for (unsigned long long x = blockIdx.x * (unsigned long long)blockDim.x + threadIdx.x; x < total;
       x += (unsigned long long)gridDim.x * blockDim.x) {
    const uint32_t r = item_request(pre_s, w.R, x);
    const uint64_t k = x - pre_s[r];
    const uint64_t s = psk::main_find(slots, ovf, tdesc[assign[r]], w.hash[w.off[r] + k]);
    if (s != ~0ull && meta.last_use[s] < last_use) meta.last_use[s] = last_use;
  }
}

__global__ void commit_insert_kernel(uint64_t* slots, uint64_t* ovf, const psk::TableDesc* __restrict__ tdesc,
                                     unsigned long long* count, psk::WindowDev w, const int32_t* __restrict__ assign,
                                     const uint32_t* __restrict__ hit_chosen, const unsigned long long* __restrict__ pre_i,
                                     psk::LruMeta meta, uint32_t last_use, uint32_t* err) {
  const unsigned long long total = pre_i[w.R];
  for (unsigned long long x = blockIdx.x * (unsigned long long)blockDim.x + threadIdx.x; x < total;
       x += (unsigned long long)gridDim.x * blockDim.x) {
    const uint32_t r = item_request(pre_i, w.R, x);
    const int32_t j = assign[r];
    const uint64_t k = hit_chosen[r] + (x - pre_i[r]);
    const uint64_t key = w.hash[w.off[r] + k];
    if (key == psk::kEmpty || key == psk::kTomb) continue;
    bool ins = false;
    const uint64_t slot = psk::thread_insert(slots, ovf, tdesc[j], key, &ins);
    if (slot == ~0ull) {
      atomicOr(err, psk::kErrTableFull);
      continue;
    }
    if (ins) {
      atomicAdd(count + j, 1ull);
      if (meta.last_use) {
        meta.last_use[slot] = last_use;
        meta.children[slot] = 0;
        meta.parent[slot] = psk::kLinkPending;
      }
    } else if (meta.last_use && meta.last_use[slot] < last_use) {
      meta.last_use[slot] = last_use;
    }
  }
}

__global__ void commit_link_kernel(const uint64_t* slots, const uint64_t* ovf, const psk::TableDesc* __restrict__ tdesc,
                                   psk::WindowDev w, const int32_t* __restrict__ assign,
                                   const uint32_t* __restrict__ hit_chosen, const unsigned long long* __restrict__ pre_i,
                                   psk::LruMeta meta) {
  const unsigned long long total = pre_i[w.R];
  for (unsigned long long x = blockIdx.x * (unsigned long long)blockDim.x + threadIdx.x; x < total;
       x += (unsigned long long)gridDim.x * blockDim.x) {
    const uint32_t r = item_request(pre_i, w.R, x);
    const psk::TableDesc d = tdesc[assign[r]];
    const uint64_t o = w.off[r];
    const uint64_t k = hit_chosen[r] + (x - pre_i[r]);
    const uint64_t key = w.hash[o + k];
    const uint64_t pkey = k > 0 ? w.hash[o + k - 1] : psk::kEmpty;
    const uint64_t s = psk::main_find(slots, ovf, d, key);
    if (s == ~0ull || meta.parent[s] != psk::kLinkPending) continue;  // not inserted by this commit
    const uint64_t ps = k > 0 ? psk::main_find(slots, ovf, d, pkey) : ~0ull;
    meta.parent[s] = ps == ~0ull ? psk::kNoParent : ps;
    if (ps != ~0ull) atomicAdd(meta.children + ps, 1u);
  }
}

__global__ void commit_queue_kernel(uint32_t I, psk::WindowDev w, const int32_t* __restrict__ assign,
                                    const uint32_t* __restrict__ hit_chosen, psk::ReqStore rq,
                                    const uint32_t* __restrict__ out_tokens, uint32_t* err) {
  const int lane = threadIdx.x & 31;
  const uint32_t warps_total = (gridDim.x * blockDim.x) >> 5;
  for (uint32_t i = (blockIdx.x * blockDim.x + threadIdx.x) >> 5; i < I; i += warps_total) {
    bool overflow = false;
    for (uint32_t r0 = 0; r0 < w.R; r0 += 32) {
      const uint32_t r = r0 + lane;
      unsigned mine = __ballot_sync(0xffffffffu, r < w.R && assign[r] == (int32_t)i);
      while (mine) {  // in arrival order
        const uint32_t rr = r0 + (uint32_t)(__ffs(mine) - 1);
        mine &= mine - 1;
        if (lane == 0) {
          const uint32_t len = rq.q_len[i];
          if (len >= rq.M) {
            overflow = true;
          } else {
            const uint64_t at = (uint64_t)i * rq.M + (rq.q_head[i] + len) % rq.M;
            rq.q_L[at] = w.L[rr];
            rq.q_out[at] = out_tokens ? out_tokens[rr] : 0u;
            rq.q_rem[at] = (uint64_t)((int64_t)w.L[rr] - 16 * (int64_t)hit_chosen[rr]);
            rq.q_len[i] = len + 1;
          }
        }
        __syncwarp();
      }
    }
    if (lane == 0 && overflow) atomicOr(err, psk::kErrRequestsFull);
  }
}

// Engine progress of one streaming window, one warp per instance (the serving engine's rules):
// every decoding request emits k = max(1, floor(window_ms / ((b0 + b1 b) + b2 S))) tokens (fp32,
// state at the window start), finished requests leave (b -= 1, S -= L + out), then the FIFO queue
// drains prefill_tokens tokens and requests whose prefill completes start decoding.
__global__ void advance_kernel(psk::StateSoA st, uint32_t I, psk::ReqStore rq, psk::DevModel m, float window_ms,
                               uint64_t prefill_tokens, uint32_t* err) {
  const int lane = threadIdx.x & 31;
  const uint32_t warps_total = (gridDim.x * blockDim.x) >> 5;
  for (uint32_t i = (blockIdx.x * blockDim.x + threadIdx.x) >> 5; i < I; i += warps_total) {
    int32_t b = st.b[i], qr = st.qr[i];
    int64_t q = st.q[i], S = st.S[i];
    float t_iter = __fadd_rn(m.b0, __fmul_rn(m.b1, __int2float_rn(b)));
    t_iter = __fadd_rn(t_iter, __fmul_rn(m.b2, __ll2float_rn(S)));
    const float per = __fdiv_rn(window_ms, t_iter);
    int64_t kk = (int64_t)per;  // per > 0: truncation is floor
    if (kk < 1) kk = 1;
    const uint32_t k = kk > 0xFFFFFFFFll ? 0xFFFFFFFFu : (uint32_t)kk;
    // decode progress with in-warp compaction of the survivors
    const uint32_t n = rq.d_len[i];
    const uint64_t base = (uint64_t)i * rq.M;
    uint32_t kept = 0;
    int64_t dS = 0;
    int32_t done = 0;
    for (uint32_t x0 = 0; x0 < n; x0 += 32) {
      const uint32_t x = x0 + lane;
      uint32_t L = 0, out = 0, rem = 0;
      bool live = false;
      if (x < n) {
        L = rq.d_L[base + x];
        out = rq.d_out[base + x];
        rem = rq.d_rem[base + x];
        const uint32_t e = rem < k ? rem : k;
        rem -= e;
        dS += e;
        live = rem > 0;
        if (!live) {
          done += 1;
          dS -= (int64_t)L + (int64_t)out;
        }
      }
      const unsigned lv = __ballot_sync(0xffffffffu, live);
      __syncwarp();
      if (live) {
        const uint32_t at = kept + __popc(lv & ((1u << lane) - 1u));
        rq.d_L[base + at] = L;
        rq.d_out[base + at] = out;
        rq.d_rem[base + at] = rem;
      }
      kept += __popc(lv);
      __syncwarp();
    }
#pragma unroll
    for (int s = 16; s > 0; s >>= 1) {
      dS += __shfl_xor_sync(0xffffffffu, dS, s);
      done += __shfl_xor_sync(0xffffffffu, done, s);
    }
    S += dS;
    b -= done;
    if (lane == 0) {
      uint32_t len = rq.q_len[i], head = rq.q_head[i];
      uint64_t budget = prefill_tokens;
      uint32_t dl = kept;
      bool overflow = false;
      while (budget > 0 && len > 0) {
        const uint64_t at = base + head;
        const uint64_t rem = rq.q_rem[at];
        const uint64_t take = rem < budget ? rem : budget;
        rq.q_rem[at] = rem - take;
        q -= (int64_t)take;
        budget -= take;
        if (rem == take) {
          if (dl < rq.M) {
            rq.d_L[base + dl] = rq.q_L[at];
            rq.d_out[base + dl] = rq.q_out[at];
            rq.d_rem[base + dl] = rq.q_out[at];
            ++dl;
          } else {
            overflow = true;
          }
          head = (head + 1) % rq.M;
          --len;
          qr -= 1;
          b += 1;
        }
      }
      rq.q_len[i] = len;
      rq.q_head[i] = head;
      rq.d_len[i] = dl;
      st.b[i] = b;
      st.qr[i] = qr;
      st.q[i] = q;
      st.S[i] = S;
      if (overflow) atomicOr(err, psk::kErrRequestsFull);
    }
  }
}

// Leaf-first LRU eviction of the instances over capacity, in rounds of two kernels:
//   collect  all SMs scan the over-capacity instances' slots (coalesced) and append each leaf (a
//            cached block with no cached child) to its instance's leaf buffer;
//   evict    one thread block per over-capacity instance sorts its leaves by (last_use, hash), then
//            thread 0 evicts in order, taking the smaller of the next sorted leaf and the smallest
//            parent that became a leaf (a small heap); the parent is reached through its stored slot.
// Every evicted block only ever makes its parent a leaf, and a leaf outside the first E sorted ones
// can never be among E evictions, so a round of at most kHeapMax evictions reproduces the
// one-at-a-time rule exactly; the host repeats rounds while an instance is still over capacity.
//
// A loader warp reads each parent's metadata from global memory ahead of the ordered loop: for the
// sorted leaves, up to kRing leaves past the loop's position; for a parent that became a leaf, as
// soon as it is pushed.  The loop never waits for it: a record not filled yet is read by the loop
// itself, with the same result.  Children counts are not written during the loop, so every read
// sees the round's starting count; the loop keeps the decremented counts in a shared hash table,
// written back at the end of the round.  A block's metadata changes in a round only when it is
// evicted, which happens after every record that names it as a parent has been read.  Most
// evictions climb a chain (a parent goes right after its last child, when its key is below the next
// candidate's); such a step reads its record itself, since the parent's parent is known only from
// the parent's metadata.
constexpr int kLeafMax = 4096;
constexpr int kHeapMax = 1536;
constexpr int kEvictThreads = 256;
constexpr int kRing = 32;          // sorted leaves whose parent records the loader keeps ready
constexpr int kDeltaSlots = 2048;  // children counts a round changes (at most kHeapMax parents)
constexpr uint64_t kEvictWaitNs = 1000000000ull;  // bound on the loader's idle wait
static_assert(kHeapMax < kDeltaSlots, "the count table never fills");
constexpr int kCollectThreads = 256;
constexpr uint32_t kCollectSlotsPerThread = 8;

// A leaf candidate with its parent's slot (kLeafNoParent for none), so that evicting it needs no
// dependent load before the parent's metadata can be read.  Five 32-bit words (the hash split).
struct Leaf {
  uint32_t last_use;
  uint32_t slot;
  uint32_t hash_lo, hash_hi;
  uint32_t parent;
};
static_assert(sizeof(Leaf) == 20, "a leaf is five 32-bit words");
constexpr uint32_t kLeafNoParent = 0xFFFFFFFFu;

__device__ __forceinline__ uint32_t parent32(uint64_t p) {
  return (p == psk::kNoParent || p == psk::kLinkPending) ? kLeafNoParent : (uint32_t)p;
}

__device__ __forceinline__ Leaf make_leaf(uint32_t last_use, uint32_t slot, uint64_t hash, uint64_t parent) {
  return Leaf{last_use, slot, (uint32_t)hash, (uint32_t)(hash >> 32), parent32(parent)};
}

__device__ __forceinline__ bool leaf_less(const Leaf& a, const Leaf& b) {
  if (a.last_use != b.last_use) return a.last_use < b.last_use;
  return a.hash_hi != b.hash_hi ? a.hash_hi < b.hash_hi : a.hash_lo < b.hash_lo;
}

__device__ __forceinline__ void heap_push(Leaf* h, int& n, const Leaf& x) {
  int c = n++;
  h[c] = x;
  while (c > 0) {
    const int p = (c - 1) >> 1;
    if (!leaf_less(h[c], h[p])) break;
    const Leaf t = h[c];
    h[c] = h[p];
    h[p] = t;
    c = p;
  }
}

__device__ __forceinline__ Leaf heap_pop(Leaf* h, int& n) {
  const Leaf top = h[0];
  h[0] = h[--n];
  int c = 0;
  for (;;) {
    const int l = 2 * c + 1, r = l + 1;
    int m = c;
    if (l < n && leaf_less(h[l], h[m])) m = l;
    if (r < n && leaf_less(h[r], h[m])) m = r;
    if (m == c) break;
    const Leaf t = h[c];
    h[c] = h[m];
    h[m] = t;
    c = m;
  }
  return top;
}

// A parent's metadata as the loader reads it: children count at the start of the round, last_use,
// hash and its own parent's slot.  A pool record also holds the slot it describes (a parent that
// became a leaf names its record by index, in the heap entry's parent word).
struct ParentRec {
  uint32_t pc, plu, ph_lo, ph_hi, ppp;
};
struct PoolRec {
  uint32_t pp;
  ParentRec r;
};
static_assert(sizeof(ParentRec) == 20 && sizeof(PoolRec) == 24, "records are 32-bit words");

// Shared memory of an eviction block.  The sort uses all kLeafMax leaves; a round then reads only
// the first kHeapMax sorted ones, and the rest of that space holds the records and the count table.
constexpr size_t kOffPool = (size_t)kHeapMax * sizeof(Leaf);
constexpr size_t kOffRing = kOffPool + (size_t)kHeapMax * sizeof(PoolRec);
constexpr size_t kOffDKey = kOffRing + (size_t)kRing * sizeof(ParentRec);
constexpr size_t kOffDVal = kOffDKey + (size_t)kDeltaSlots * sizeof(uint32_t);
constexpr size_t kOffHeapRaw = kOffDVal + (size_t)kDeltaSlots * sizeof(uint32_t);
constexpr size_t kOffHeap =
    kOffHeapRaw > (size_t)kLeafMax * sizeof(Leaf) ? kOffHeapRaw : (size_t)kLeafMax * sizeof(Leaf);
constexpr size_t kEvictSmem = kOffHeap + (size_t)kHeapMax * sizeof(Leaf);
// two eviction blocks per SM: 2 x (kEvictSmem + the static flags + 1 KB reserved) <= 228 KB
static_assert(2 * (kEvictSmem + 64 + 1024) <= 228 * 1024, "two eviction blocks fit on an SM");
__device__ __forceinline__ ParentRec load_parent(const uint64_t* slots, const psk::LruMeta& meta, uint32_t ps) {
  ParentRec r{0u, 0u, 0u, 0u, kLeafNoParent};
  if (ps != kLeafNoParent) {
    const uint32_t pc = meta.children[ps], plu = meta.last_use[ps];
    const uint64_t ph = slots[ps], pp = meta.parent[ps];
    r = ParentRec{pc, plu, (uint32_t)ph, (uint32_t)(ph >> 32), parent32(pp)};
  }
  return r;
}
// The decremented children count of ps (first touch: from the round's starting count pc).
__device__ __forceinline__ uint32_t count_dec(uint32_t* dkey, uint32_t* dval, uint32_t ps, uint32_t pc) {
  uint32_t h = (ps * 0x9E3779B1u) >> 21;  // 11 bits: kDeltaSlots entries
  for (int probe = 0; probe < kDeltaSlots; ++probe) {
    const uint32_t k = dkey[h];
    if (k == ps) return --dval[h];
    if (k == kLeafNoParent) {
      dkey[h] = ps;
      dval[h] = pc - 1u;
      return pc - 1u;
    }
    h = (h + 1u) & (uint32_t)(kDeltaSlots - 1);
  }
  return 1u;  // not reached: a round changes fewer counts than the table holds
}
static_assert(kDeltaSlots == 1 << 11, "count_dec hashes to 11 bits");

struct EvictFlags {
  uint32_t ptr;        // sorted leaves the loop has taken (their records may be overwritten)
  uint32_t ring_done;  // sorted leaves whose parent records are in the ring
  uint32_t req;        // pool records the loop has asked for
  uint32_t pool_done;  // pool records filled
  uint32_t exit;       // the loop has ended
};

// The loader warp: fills ring records for sorted leaves [ring_done, min(m, ptr + kRing)) and pool
// records [pool_done, req), one record of each kind per lane per pass, loads issued before any
// record is written.  Every control value is the warp's minimum of what its lanes observed, so the
// warp stays converged and each lane's acquire covers what it reads.
__device__ void evict_loader(const uint64_t* slots, const psk::LruMeta& meta, const Leaf* leaves, ParentRec* ring,
                             PoolRec* pool, uint32_t m, EvictFlags* f, uint32_t* err) {
  const uint32_t lane = threadIdx.x & 31u;
  uint32_t ring_done = 0, pool_done = 0;
  const long long c0 = clock64();
  const long long lim = (long long)(kEvictWaitNs * 3ull);
  for (uint32_t it = 1;; ++it) {
    uint32_t ex = psk::ld_relaxed_cta_shared_u32(&f->exit);
    uint32_t ptr = psk::ld_relaxed_cta_shared_u32(&f->ptr);
    uint32_t req = psk::ld_relaxed_cta_shared_u32(&f->req);
    psk::fence_acq_rel_cta();
    ex = __reduce_min_sync(0xffffffffu, ex);
    ptr = __reduce_min_sync(0xffffffffu, ptr);
    req = __reduce_min_sync(0xffffffffu, req);
    if (ex) return;
    const uint32_t rhi = ptr + (uint32_t)kRing < m ? ptr + (uint32_t)kRing : m;
    const uint32_t phi = req < pool_done + 32u ? req : pool_done + 32u;
    if (ring_done >= rhi && pool_done >= phi) {
      if ((it & 31u) == 0u && __any_sync(0xffffffffu, clock64() - c0 > lim)) {
        if (lane == 0) atomicOr(err, psk::kErrTimeout);
        return;
      }
      continue;
    }
    const uint32_t j = ring_done + lane, k = pool_done + lane;
    const bool rj = j < rhi, pk = k < phi;
    const ParentRec a = load_parent(slots, meta, rj ? leaves[j].parent : kLeafNoParent);
    const uint32_t pp = pk ? pool[k].pp : kLeafNoParent;
    const ParentRec b = load_parent(slots, meta, pp);
    if (rj) ring[j % (uint32_t)kRing] = a;
    if (pk) pool[k].r = b;
    __syncwarp();
    if (lane == 0) {
      if (rhi > ring_done) psk::st_release_cta_shared_u32(&f->ring_done, rhi);
      if (phi > pool_done) psk::st_release_cta_shared_u32(&f->pool_done, phi);
    }
    if (rhi > ring_done) ring_done = rhi;
    if (phi > pool_done) pool_done = phi;
  }
}

// grid: (slot chunks, instances)
__global__ void __launch_bounds__(kCollectThreads)
leaf_collect_kernel(const uint64_t* __restrict__ slots, const psk::TableDesc* __restrict__ tdesc,
                    const unsigned long long* __restrict__ count, const uint64_t* __restrict__ cap, psk::LruMeta meta,
                    Leaf* __restrict__ leafbuf, uint32_t* __restrict__ nleaf) {
  const uint32_t i = blockIdx.y;
  if (count[i] <= cap[i]) return;  // block-uniform
  const psk::TableDesc d = tdesc[i];
  const uint64_t nslots = (uint64_t)d.nbkt * psk::kBucketSlots;
  const uint64_t stride = (uint64_t)gridDim.x * kCollectThreads;
  for (uint64_t x = (uint64_t)blockIdx.x * kCollectThreads + threadIdx.x; x < nslots; x += stride) {
    const uint64_t s = d.base + x;
    const uint64_t key = __ldcs(slots + s);
    if (key == psk::kEmpty || key == psk::kTomb || meta.children[s] != 0u) continue;
    const uint32_t at = atomicAdd(nleaf + i, 1u);
    if (at < (uint32_t)kLeafMax)
      leafbuf[(uint64_t)i * kLeafMax + at] = make_leaf(meta.last_use[s], (uint32_t)s, key, meta.parent[s]);
  }
}

__global__ void __launch_bounds__(kEvictThreads)
evict_kernel(uint64_t* slots, unsigned long long* count, const uint64_t* __restrict__ cap, psk::LruMeta meta,
             const Leaf* __restrict__ leafbuf, const uint32_t* __restrict__ nleaf, uint32_t* more, uint32_t* err) {
  extern __shared__ __align__(16) unsigned char ev_smem[];
  __shared__ EvictFlags flags;
  Leaf* leaves = reinterpret_cast<Leaf*>(ev_smem);
  PoolRec* pool = reinterpret_cast<PoolRec*>(ev_smem + kOffPool);
  ParentRec* ring = reinterpret_cast<ParentRec*>(ev_smem + kOffRing);
  uint32_t* dkey = reinterpret_cast<uint32_t*>(ev_smem + kOffDKey);
  uint32_t* dval = reinterpret_cast<uint32_t*>(ev_smem + kOffDVal);
  Leaf* heap = reinterpret_cast<Leaf*>(ev_smem + kOffHeap);
  const uint32_t i = blockIdx.x;
  const unsigned long long cnt = count[i];
  if (cnt <= cap[i]) return;  // block-uniform
  // an earlier round gave up: no more rounds (read once, so that the whole block leaves together)
  if (__syncthreads_or(threadIdx.x == 0 && (*(volatile uint32_t*)err & psk::kErrTimeout) != 0u)) return;
  const uint32_t n = nleaf[i];
  if (n > (uint32_t)kLeafMax || n == 0) {
    if (threadIdx.x == 0) atomicOr(err, psk::kErrLeavesFull);
    return;
  }
  uint32_t np2 = 1;
  while (np2 < n) np2 <<= 1;
  for (uint32_t x = threadIdx.x; x < np2; x += kEvictThreads)
    leaves[x] = x < n ? leafbuf[(uint64_t)i * kLeafMax + x]
                      : Leaf{0xFFFFFFFFu, 0xFFFFFFFFu, 0xFFFFFFFFu, 0xFFFFFFFFu, kLeafNoParent};
  __syncthreads();
  for (uint32_t size = 2; size <= np2; size <<= 1) {  // bitonic sort by (last_use, hash)
    for (uint32_t stride = size >> 1; stride > 0; stride >>= 1) {
      for (uint32_t x = threadIdx.x; x < np2; x += kEvictThreads) {
        const uint32_t y = x ^ stride;
        if (y > x) {
          const bool up = (x & size) == 0;
          const Leaf a = leaves[x], b = leaves[y];
          if (leaf_less(b, a) == up) {
            leaves[x] = b;
            leaves[y] = a;
          }
        }
      }
      __syncthreads();
    }
  }
  const uint64_t E = cnt - cap[i];
  const uint32_t todo = E < (uint64_t)kHeapMax ? (uint32_t)E : (uint32_t)kHeapMax;
  const uint32_t m = n < todo ? n : todo;  // sorted leaves a round can take
  for (uint32_t x = threadIdx.x; x < (uint32_t)kDeltaSlots; x += kEvictThreads) dkey[x] = kLeafNoParent;
  if (threadIdx.x == 0) flags = EvictFlags{0u, 0u, 0u, 0u, 0u};
  __syncthreads();
  const uint32_t warp = threadIdx.x >> 5;
  if (warp >= 2) return;
  if (warp == 1) {
    evict_loader(slots, meta, leaves, ring, pool, m, &flags, err);
  } else if (threadIdx.x == 0) {
    uint32_t ptr = 0, npush = 0;
    int hn = 0;
    uint32_t evicted = 0;
    while (evicted < todo) {
      const bool from_sorted = ptr < n && (hn == 0 || leaf_less(leaves[ptr], heap[0]));
      if (!from_sorted && hn == 0) break;
      Leaf v;
      uint32_t ps = kLeafNoParent;
      ParentRec r{0u, 0u, 0u, 0u, kLeafNoParent};
      if (from_sorted) {
        v = leaves[ptr];
        ps = v.parent;
        if (ps != kLeafNoParent) {
          if (psk::ld_relaxed_cta_shared_u32(&flags.ring_done) > ptr) {
            psk::fence_acq_rel_cta();
            r = ring[ptr % (uint32_t)kRing];
          } else {
            r = load_parent(slots, meta, ps);
          }
        }
        ++ptr;
        psk::st_release_cta_shared_u32(&flags.ptr, ptr);  // the record is read: its slot may be refilled
      } else {
        v = heap_pop(heap, hn);
        if (v.parent != kLeafNoParent) {
          ps = pool[v.parent].pp;
          if (psk::ld_relaxed_cta_shared_u32(&flags.pool_done) > v.parent) {
            psk::fence_acq_rel_cta();
            r = pool[v.parent].r;
          } else {
            r = load_parent(slots, meta, ps);
          }
        }
      }
      slots[v.slot] = psk::kEmpty;
      meta.last_use[v.slot] = 0;
      meta.children[v.slot] = 0;
      meta.parent[v.slot] = psk::kNoParent;
      ++evicted;
      if (ps != kLeafNoParent && count_dec(dkey, dval, ps, r.pc) == 0u) {
        uint32_t link = kLeafNoParent;
        if (r.ppp != kLeafNoParent) {  // ask the loader for the record of its parent
          link = npush;
          pool[npush].pp = r.ppp;
          psk::st_release_cta_shared_u32(&flags.req, ++npush);
        }
        heap_push(heap, hn, Leaf{r.plu, ps, r.ph_lo, r.ph_hi, link});
      }
    }
    count[i] = cnt - evicted;
    if (evicted > 0 && cnt - evicted > cap[i]) atomicOr(more, 1u);
    psk::st_release_cta_shared_u32(&flags.exit, 1u);
  }
  __syncwarp();
  asm volatile("bar.sync 1, 64;" ::: "memory");  // warps 0 and 1: the loop and the loader are done
  for (uint32_t x = threadIdx.x; x < (uint32_t)kDeltaSlots; x += 64u)
    if (dkey[x] != kLeafNoParent) meta.children[dkey[x]] = dval[x];
}

// Prefix closure check (search mode): every chain's parent must be cached once the chains are in.
__global__ void check_parents_kernel(const uint64_t* slots, const uint64_t* ovf, const psk::TableDesc* __restrict__ tdesc, uint32_t I,
                                     uint64_t nchains, const uint32_t* __restrict__ inst,
                                     const uint64_t* __restrict__ parent, uint32_t* err) {
  for (uint64_t c = blockIdx.x * (uint64_t)blockDim.x + threadIdx.x; c < nchains; c += (uint64_t)gridDim.x * blockDim.x) {
    const uint64_t p = parent[c];
    const uint32_t i = inst[c];
    if (p == psk::kEmpty || i >= I) continue;
    if (!psk::main_contains(slots, ovf, tdesc[i], p)) atomicOr(err, psk::kErrParentMissing);
  }
}

__global__ void validate_window_kernel(psk::WindowDev w, uint64_t max_blocks, uint32_t* err) {
  for (uint32_t r = blockIdx.x * blockDim.x + threadIdx.x; r < w.R; r += gridDim.x * blockDim.x) {
    const uint64_t a = w.off[r], b = w.off[r + 1];
    const uint32_t L = w.L[r];
    bool ok = b >= a && (b - a) == (uint64_t)(L / 16u) && L < (1u << 30) && b <= max_blocks;
    if (r == 0) ok = ok && a == 0;
    if (!ok) atomicOr(err, psk::kErrWindowLayout);
  }
}

}  // namespace

namespace pskl {

cudaError_t launch_insert_chains(uint64_t* slots, uint64_t* ovf, const psk::TableDesc* tdesc, uint32_t I,
                                 unsigned long long* count, uint64_t nchains, const uint32_t* inst,
                                 const uint64_t* off, const uint64_t* hash, const uint64_t* parent,
                                 uint64_t total, psk::LruMeta meta, uint32_t last_use, uint32_t* err,
                                 int num_sms, cudaStream_t s) {
  if (total == 0 || nchains == 0) return cudaSuccess;
  uint64_t blocks = (nchains + 255) / 256;
  if (blocks > (uint64_t)num_sms * 8) blocks = (uint64_t)num_sms * 8;
  check_instances_kernel<<<(unsigned)blocks, 256, 0, s>>>(I, nchains, inst, err);
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  const uint32_t warps_per_block = 4;
  insert_chains_kernel<<<(I + warps_per_block - 1) / warps_per_block, 32 * warps_per_block, 0, s>>>(
      slots, ovf, tdesc, I, count, nchains, inst, off, hash, parent, meta, last_use, err);
  return cudaGetLastError();
}

cudaError_t launch_commit(uint64_t* slots, uint64_t* ovf, const psk::TableDesc* tdesc, uint32_t I,
                          unsigned long long* count, const psk::WindowDev& w, const int32_t* assign,
                          const uint32_t* hit_chosen, psk::LruMeta meta, uint32_t last_use,
                          const psk::ReqStore& rq, const uint32_t* out_tokens, unsigned long long* prefix,
                          uint32_t* err, int num_sms, cudaStream_t s) {
  if (w.R == 0) return cudaSuccess;
  unsigned long long* pre_s = prefix;          // [R + 1]
  unsigned long long* pre_i = prefix + w.R + 1;  // [R + 1]
  commit_prefix_kernel<<<1, 1024, 0, s>>>(w, assign, hit_chosen, pre_s, pre_i);
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  const uint32_t g = (uint32_t)num_sms * 8u;  // flat items, grid-stride
  if (meta.last_use) {
    commit_stamp_kernel<<<g, 256, 0, s>>>(slots, ovf, tdesc, w, assign, pre_s, meta, last_use);
    e = cudaGetLastError();
    if (e != cudaSuccess) return e;
  }
  commit_insert_kernel<<<g, 256, 0, s>>>(slots, ovf, tdesc, count, w, assign, hit_chosen, pre_i, meta, last_use, err);
  e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  if (meta.last_use) {
    commit_link_kernel<<<g, 256, 0, s>>>(slots, ovf, tdesc, w, assign, hit_chosen, pre_i, meta);
    e = cudaGetLastError();
    if (e != cudaSuccess) return e;
  }
  if (rq.M) {
    const uint32_t warps_per_block = 4;
    commit_queue_kernel<<<(I + warps_per_block - 1) / warps_per_block, 32 * warps_per_block, 0, s>>>(
        I, w, assign, hit_chosen, rq, out_tokens, err);
    e = cudaGetLastError();
  }
  return e;
}

cudaError_t launch_advance(psk::StateSoA st, uint32_t I, const psk::ReqStore& rq, const psk::DevModel& m,
                           float window_ms, uint64_t prefill_tokens, uint32_t* err, cudaStream_t s) {
  const uint32_t warps_per_block = 4;
  advance_kernel<<<(I + warps_per_block - 1) / warps_per_block, 32 * warps_per_block, 0, s>>>(
      st, I, rq, m, window_ms, prefill_tokens, err);
  return cudaGetLastError();
}

cudaError_t launch_evict(uint64_t* slots, const psk::TableDesc* tdesc, uint32_t I, unsigned long long* count,
                         const uint64_t* cap, psk::LruMeta meta, void* leafbuf, uint32_t* nleaf, uint32_t* more,
                         uint32_t* more_host, uint64_t max_instance_slots, uint32_t* err, cudaStream_t s) {
  const size_t smem = kEvictSmem;
  cudaError_t e = cudaFuncSetAttribute(evict_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (e != cudaSuccess) return e;
  const uint64_t per_block = (uint64_t)kCollectThreads * kCollectSlotsPerThread;
  const unsigned gx = (unsigned)((max_instance_slots + per_block - 1) / per_block);
  for (int round = 0; round < 4096; ++round) {
    if ((e = cudaMemsetAsync(nleaf, 0, (size_t)I * sizeof(uint32_t), s)) != cudaSuccess) return e;
    if ((e = cudaMemsetAsync(more, 0, sizeof(uint32_t), s)) != cudaSuccess) return e;
    leaf_collect_kernel<<<dim3(gx ? gx : 1u, I), kCollectThreads, 0, s>>>(slots, tdesc, count, cap, meta,
                                                                           static_cast<Leaf*>(leafbuf), nleaf);
    if ((e = cudaGetLastError()) != cudaSuccess) return e;
    evict_kernel<<<I, kEvictThreads, smem, s>>>(slots, count, cap, meta, static_cast<const Leaf*>(leafbuf), nleaf,
                                                more, err);
    if ((e = cudaGetLastError()) != cudaSuccess) return e;
    if ((e = cudaMemcpyAsync(more_host, more, sizeof(uint32_t), cudaMemcpyDeviceToHost, s)) != cudaSuccess) return e;
    if ((e = cudaStreamSynchronize(s)) != cudaSuccess) return e;
    if (*more_host == 0u) break;
  }
  return cudaSuccess;
}

size_t evict_leafbuf_bytes(uint32_t I) { return (size_t)I * kLeafMax * sizeof(Leaf); }

cudaError_t launch_check_parents(const uint64_t* slots, const uint64_t* ovf, const psk::TableDesc* tdesc, uint32_t I,
                                 uint64_t nchains, const uint32_t* inst, const uint64_t* parent,
                                 uint32_t* err, int num_sms, cudaStream_t s) {
  if (nchains == 0) return cudaSuccess;
  uint64_t blocks = (nchains + 255) / 256;
  if (blocks > (uint64_t)num_sms * 8) blocks = (uint64_t)num_sms * 8;
  check_parents_kernel<<<(unsigned)blocks, 256, 0, s>>>(slots, ovf, tdesc, I, nchains, inst, parent, err);
  return cudaGetLastError();
}

cudaError_t launch_validate_window(const psk::WindowDev& w, uint64_t max_blocks, uint32_t* err,
                                   cudaStream_t s) {
  if (w.R == 0) return cudaSuccess;
  uint32_t blocks = (w.R + 255) / 256;
  if (blocks > 1024) blocks = 1024;
  validate_window_kernel<<<blocks, 256, 0, s>>>(w, max_blocks, err);
  return cudaGetLastError();
}

}  // namespace pskl
