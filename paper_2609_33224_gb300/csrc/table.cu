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

// Commit: one warp per instance applies that instance's admitted requests in arrival order: the
// cached prefix chain[0..h) is stamped last_use (lanes in parallel), the uncached blocks
// chain[h..nb) are cached (stamped, parents linked), and with request tracking the request joins
// the instance's FIFO queue with its uncached tokens as remaining prefill.
__global__ void commit_kernel(uint64_t* slots, uint64_t* ovf, const psk::TableDesc* __restrict__ tdesc, uint32_t I,
                              unsigned long long* count, psk::WindowDev w, const int32_t* __restrict__ assign,
                              const uint32_t* __restrict__ hit_chosen, psk::LruMeta meta, uint32_t last_use,
                              psk::ReqStore rq, const uint32_t* __restrict__ out_tokens, uint32_t* err) {
  const int lane = threadIdx.x & 31;
  const uint32_t warps_total = (gridDim.x * blockDim.x) >> 5;
  for (uint32_t i = (blockIdx.x * blockDim.x + threadIdx.x) >> 5; i < I; i += warps_total) {
    const psk::TableDesc d = tdesc[i];
    unsigned long long added = 0;
    bool full = false, overflow = false;
    for (uint32_t r0 = 0; r0 < w.R; r0 += 32) {
      const uint32_t r = r0 + lane;
      unsigned mine = __ballot_sync(0xffffffffu, r < w.R && assign[r] == (int32_t)i);
      while (mine) {
        const int l = __ffs(mine) - 1;
        mine &= mine - 1;
        const uint32_t rr = r0 + l;
        const uint64_t o = w.off[rr];
        const uint64_t nb = w.off[rr + 1] - o;
        const uint64_t h = hit_chosen[rr];
        if (meta.last_use) {
          for (uint64_t k = lane; k < h; k += 32) {
            const uint64_t s = psk::main_find(slots, ovf, d, w.hash[o + k]);
            if (s != ~0ull && meta.last_use[s] < last_use) meta.last_use[s] = last_use;
          }
          __syncwarp();
        }
        uint64_t prev_key = h ? w.hash[o + h - 1] : psk::kEmpty, prev_slot = ~0ull;
        for (uint64_t k = h; k < nb && !full; ++k) {
          const uint64_t key = w.hash[o + k];
          if (key == psk::kEmpty || key == psk::kTomb) {
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
        if (rq.M && lane == 0) {
          const uint32_t len = rq.q_len[i];
          if (len >= rq.M) {
            overflow = true;
          } else {
            const uint64_t at = (uint64_t)i * rq.M + (rq.q_head[i] + len) % rq.M;
            rq.q_L[at] = w.L[rr];
            rq.q_out[at] = out_tokens ? out_tokens[rr] : 0u;
            rq.q_rem[at] = (uint64_t)((int64_t)w.L[rr] - 16 * (int64_t)h);
            rq.q_len[i] = len + 1;
          }
        }
        __syncwarp();
      }
    }
    if (lane == 0) {
      count[i] += added;
      if (full) atomicOr(err, psk::kErrTableFull);
      if (overflow) atomicOr(err, psk::kErrRequestsFull);
    }
  }
}

// Engine progress of one streaming window, one warp per instance (the rules the oracle states):
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

// Leaf-first LRU eviction, one thread block per instance over capacity.  Per round: collect the
// instance's leaves (cached blocks with no cached child) into shared memory, sort them by
// (last_use, hash), then thread 0 evicts in order, taking the smaller of the next sorted leaf and the
// smallest parent that became a leaf (a small heap).  Every evicted block only ever makes its parent
// a leaf, and a leaf outside the first E sorted ones can never be among E evictions, so a round of
// at most kHeapMax evictions reproduces the one-at-a-time rule exactly; rounds repeat until the
// instance is at capacity.
constexpr int kLeafMax = 4096;
constexpr int kHeapMax = 2048;
constexpr int kEvictThreads = 256;

struct Leaf {
  uint32_t last_use;
  uint32_t pad;
  uint64_t hash;
  uint64_t slot;
};

__device__ __forceinline__ bool leaf_less(const Leaf& a, const Leaf& b) {
  return a.last_use != b.last_use ? a.last_use < b.last_use : a.hash < b.hash;
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

__global__ void __launch_bounds__(kEvictThreads)
evict_kernel(uint64_t* slots, uint64_t* ovf, const psk::TableDesc* __restrict__ tdesc, uint32_t I,
             unsigned long long* count, const uint64_t* __restrict__ cap, psk::LruMeta meta, uint32_t* err) {
  extern __shared__ unsigned long long ev_smem[];
  Leaf* leaves = reinterpret_cast<Leaf*>(ev_smem);
  Leaf* heap = leaves + kLeafMax;
  __shared__ uint32_t s_nleaf;
  __shared__ int s_stop;
  for (uint32_t i = blockIdx.x; i < I; i += gridDim.x) {
    const psk::TableDesc d = tdesc[i];
    const uint64_t nslots = (uint64_t)d.nbkt * psk::kBucketSlots;
    for (;;) {
      const unsigned long long cnt = count[i];
      if (cnt <= cap[i]) break;
      const uint64_t E = cnt - cap[i];
      if (threadIdx.x == 0) {
        s_nleaf = 0;
        s_stop = 0;
      }
      __syncthreads();
      for (uint64_t x = threadIdx.x; x < nslots; x += kEvictThreads) {
        const uint64_t s = d.base + x;
        const uint64_t key = slots[s];
        if (key != psk::kEmpty && meta.children[s] == 0) {
          const uint32_t at = atomicAdd(&s_nleaf, 1u);
          if (at < kLeafMax) leaves[at] = Leaf{meta.last_use[s], 0u, key, s};
        }
      }
      __syncthreads();
      const uint32_t nleaf = s_nleaf;
      if (nleaf > kLeafMax || nleaf == 0) {
        if (threadIdx.x == 0) atomicOr(err, psk::kErrLeavesFull);
        break;
      }
      // bitonic sort of the leaves (padded to a power of two with +infinity)
      uint32_t np2 = 1;
      while (np2 < nleaf) np2 <<= 1;
      for (uint32_t x = nleaf + threadIdx.x; x < np2; x += kEvictThreads)
        leaves[x] = Leaf{0xFFFFFFFFu, 0u, ~0ull, ~0ull};
      __syncthreads();
      for (uint32_t size = 2; size <= np2; size <<= 1) {
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
      if (threadIdx.x == 0) {
        const uint64_t todo = E < (uint64_t)kHeapMax ? E : (uint64_t)kHeapMax;
        uint32_t ptr = 0;
        int hn = 0;
        uint64_t evicted = 0;
        while (evicted < todo) {
          const bool from_sorted = ptr < nleaf && (hn == 0 || leaf_less(leaves[ptr], heap[0]));
          if (!from_sorted && hn == 0) break;
          const Leaf v = from_sorted ? leaves[ptr++] : heap_pop(heap, hn);
          const uint64_t parent = meta.parent[v.slot];
          slots[v.slot] = psk::kEmpty;
          meta.last_use[v.slot] = 0;
          meta.children[v.slot] = 0;
          meta.parent[v.slot] = 0;
          ++evicted;
          if (parent != psk::kEmpty) {
            const uint64_t ps = psk::main_find(slots, ovf, d, parent);
            if (ps != ~0ull) {
              const uint32_t c = meta.children[ps] - 1;
              meta.children[ps] = c;
              if (c == 0) heap_push(heap, hn, Leaf{meta.last_use[ps], 0u, parent, ps});
            }
          }
        }
        count[i] = cnt - evicted;
        if (evicted == 0) s_stop = 1;
      }
      __syncthreads();
      if (s_stop) break;
    }
    __syncthreads();
  }
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
                          const psk::ReqStore& rq, const uint32_t* out_tokens, uint32_t* err, int num_sms,
                          cudaStream_t s) {
  (void)num_sms;
  if (w.R == 0) return cudaSuccess;
  const uint32_t warps_per_block = 4;
  commit_kernel<<<(I + warps_per_block - 1) / warps_per_block, 32 * warps_per_block, 0, s>>>(
      slots, ovf, tdesc, I, count, w, assign, hit_chosen, meta, last_use, rq, out_tokens, err);
  return cudaGetLastError();
}

cudaError_t launch_advance(psk::StateSoA st, uint32_t I, const psk::ReqStore& rq, const psk::DevModel& m,
                           float window_ms, uint64_t prefill_tokens, uint32_t* err, cudaStream_t s) {
  const uint32_t warps_per_block = 4;
  advance_kernel<<<(I + warps_per_block - 1) / warps_per_block, 32 * warps_per_block, 0, s>>>(
      st, I, rq, m, window_ms, prefill_tokens, err);
  return cudaGetLastError();
}

cudaError_t launch_evict(uint64_t* slots, uint64_t* ovf, const psk::TableDesc* tdesc, uint32_t I,
                         unsigned long long* count, const uint64_t* cap, psk::LruMeta meta, uint32_t* err,
                         cudaStream_t s) {
  const size_t smem = (size_t)(kLeafMax + kHeapMax) * sizeof(Leaf);
  cudaError_t e = cudaFuncSetAttribute(evict_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (e != cudaSuccess) return e;
  evict_kernel<<<I, kEvictThreads, smem, s>>>(slots, ovf, tdesc, I, count, cap, meta, err);
  return cudaGetLastError();
}

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
