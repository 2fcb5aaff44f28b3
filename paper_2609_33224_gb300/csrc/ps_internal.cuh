// Device-side data layout and shared device functions of the scheduler library (sm_103a).
//
// HBM layout
//   main tables   one u64 slot array for all instances; instance i owns nbkt_i buckets of 8 slots
//                 (one 64-byte half line each) starting at slot base_i.  Balanced two-choice
//                 hashing: a block hash h may live in bucket b1 = fastrange(h) or
//                 b2 = fastrange(remix(h)) and is inserted into the emptier of the two (b1 on
//                 ties).  A lookup reads both 64-byte buckets at once, so a hit or a miss costs one
//                 memory round trip.  If both buckets are full the key goes to the first non-full
//                 bucket after b1 (wrapping) and b1 plus every full bucket passed get their bit set
//                 in the instance's overflow bitmap; at load factor 0.9 about 0.6% of keys take that
//                 path.  Slot value 0 = empty.  Each table has a single writer (one warp per
//                 instance), so placement needs no atomics and a key is never stored twice.
//   delta table   window-scoped set of (instance, block) pairs cached by the window's own earlier
//                 decisions: one 16-byte slot {hash, instance + 1} per pair, linear probing from the
//                 hash's home slot, sized at twice the window's block bound so it can never fill.
//                 Cleared after each window.
//   state         structure of arrays per instance (b, qr, q, S, M_KV, B_max).
//   hits          u32 [R x I], request-major.
#pragma once

#include <cstdint>
#include <cuda_runtime.h>

namespace psk {

constexpr uint64_t kEmpty = 0ull;
constexpr uint64_t kTomb = ~0ull;
constexpr int kBucketSlots = 8;    // main table: 8 x 8 B = 64 B
constexpr uint32_t kDeltaNoInst = 0xFFFFFFFFu;

// Device error bits, OR-ed into one word per context and turned into a ps_status on the host.
enum : uint32_t {
  kErrTableFull = 1u,
  kErrReservedHash = 2u,
  kErrDeltaFull = 4u,
  kErrWindowLayout = 8u,
  kErrBadInstance = 16u,
  kErrParentMissing = 32u,
  kErrTimeout = 64u,
  kErrRequestsFull = 128u,
  kErrLeavesFull = 256u,
  kErrTableLayout = 512u,
};

struct TableDesc {
  uint64_t base;   // first slot of the instance's table
  uint64_t ovf;    // first u64 word of the instance's overflow bitmap (one bit per bucket)
  uint32_t nbkt;   // buckets
  uint32_t pad;
};

// One (block, instance) pair of the window's delta table: the block hash and instance id + 1 (0 while
// the claiming thread has not yet written it).  Within one window each pair is inserted at most once:
// a request inserts chain[h, nb) on its pick with h the exact first miss there, so none of those
// blocks is cached on that instance yet (a block hash fixes its whole prefix, so an earlier insert of
// the same block would have cached chain[0, that position] and moved the first miss past it).
struct DeltaSlot {
  unsigned long long hash;
  unsigned int tag;
  unsigned int pad;
};

// Greedy pipeline depth: a probe for request s sees every delta insert of requests <= s - kLag, and
// the requests s - 1 .. s - (kLag - 1) are covered by their common chain prefix with s (RowPre::lcp).
constexpr int kLag = 21;
constexpr int kLcpBack = kLag - 1;

// Per-request constants of one window, computed in parallel before the greedy pass: the request's
// chain range, the Algorithm 1 / Eq. 8 row constants, and its relations to earlier requests of the
// window (longest common chain prefix with each of the kLcpBack requests before it; the deepest earlier
// request whose whole chain is a prefix of this one).
struct __align__(16) RowPre {
  uint64_t off;
  uint32_t nb;
  uint32_t L;
  float t_cached;     // T_pf(0, L)
  float Z;            // T_pf(L, 0) - T_pf(0, L)
  float etaZ;         // eta * Z
  float ttft_budget;  // max(target, T_pf(L, 0))
  float tpot_target;
  int32_t par;        // deepest earlier request whose chain is a prefix of r's, -1 if none
  uint32_t par_nb;    // its chain length
  int32_t base;       // the topmost request of r's parent links (r's chain starts with its chain), -1 if none
  int32_t anc[2];     // the parent's parent and its parent (-1 if none): their chains are prefixes too
  uint32_t anc_nb[2]; // their chain lengths
  uint32_t lcp[kLcpBack];  // common chain prefix with requests r - 1 .. r - kLcpBack (blocks)
};
constexpr int kRowWords = (int)(sizeof(RowPre) / 16);
static_assert(sizeof(RowPre) % 16 == 0 && kRowWords <= 32, "RowPre is whole 16-byte words, staged by one warp");

// Hand-offs between the blocks of the pipelined greedy (one cooperative launch): the deciding
// block publishes each decision as a job, insert blocks put the job's chain blocks into the delta
// table, probe blocks turn hit0 rows into the hits the deciding block reads.
constexpr uint32_t kHitSlots = 64;  // rows of probed hits in flight (a ring; more than kLag + 2)
// Rows of a window whose hits are searched from scratch (no earlier request of the window is a
// prefix of theirs), in no particular order: filled by the relations pass, read by the probe.
struct RowList {
  uint32_t* rows;   // [R]
  uint32_t* count;  // [1]
};

// Lag-d speculation of the greedy pass: summary blocks evaluate row s in full on the state before
// decision s - kSpecLag and publish a RowSummary; the deciding warp corrects it for the instances
// picked by decisions s - kSpecLag .. s - 1 (kSpecLag <= kLcpBack, so their common chain prefixes
// with request s are in RowPre::lcp).
constexpr int kSpecLag = 8;
constexpr int kSumWarps = 8;      // warps of a summary block (256 threads)
constexpr int kKeysPerWarp = 4;   // smallest (key, tie) pairs of C a summary warp publishes
constexpr int kWPerWarp = 2;      // smallest (W, instance) pairs of A a summary warp publishes
constexpr uint32_t kSumSlots = 64;  // ring of published summaries (row s in slot s % kSumSlots)
static_assert(kSpecLag <= kLcpBack, "the corrected picks need their common prefix with the row");

// Summary of row s on the state before decision s - kSpecLag: for each of the kSumWarps warps its
// kKeysPerWarp smallest packed keys of C (with tie word, W and hit) and its kWPerWarp smallest W of A;
// every pair of C it does not publish has (key, tie) >= (key_bound, tie_bound), every W of A it does
// not publish is >= the W bound.  W values travel as order-preserving bits (f2ord).
struct __align__(16) RowSummary {
  unsigned long long key[kSumWarps * kKeysPerWarp];  // packed (class, value) keys; kNoKey: none
  uint32_t tie[kSumWarps * kKeysPerWarp];            // tie words (instance in the low 12 bits)
  uint32_t word[kSumWarps * kKeysPerWarp];           // f2ord(W) of the pair
  uint32_t hit[kSumWarps * kKeysPerWarp];            // its hit (blocks)
  unsigned long long w[kSumWarps * kWPerWarp];       // f2ord(W) << 32 | instance over A; ~0: none
  unsigned long long key_bound;                      // kNoKey: every pair of C is published
  uint32_t tie_bound;
  uint32_t w_bound;                                  // 0xFFFFFFFF: every W of A is published
  uint32_t wmin;                                     // f2ord(W_min over A), 0xFFFFFFFF: A empty
  uint32_t pad[3];
};
static_assert(sizeof(RowSummary) % 16 == 0, "summaries are copied in 16-byte pieces");

struct GreedySync {
  unsigned long long* jobs;  // [R] 1 << 63 | hit of the pick << 32 | pick (0xFFFFFFFF = rejected); 0 = unpublished
  uint32_t* done;            // [R] insert blocks done with the job (its blocks are all in at the group size)
  uint32_t* ready;           // [R] 1 once the row's probed hits are in the ring
  uint32_t* hitring;         // [kHitSlots][ring_stride] probed hits (row s in slot s % kHitSlots)
  float* tpfring;            // [kHitSlots][ring_stride] T_pf at those hits (kNoTpfBits where it changed)
  uint32_t ring_stride;      // I rounded up to a multiple of 4
  uint64_t wait_ns;          // bound on any cross-block wait (ns); a waiter that gives up sets kErrTimeout
  RowSummary* sums;          // [kSumSlots] published row summaries
  uint32_t* sready;          // [R] 1 once row s's summary is published
  unsigned long long* stats; // [kGreedyStats] counters of the pass (below)
};

// Counters of one greedy pass (GreedySync::stats): decisions taken from a corrected summary and by a
// full pass, then SM clock cycles summed over the blocks of each role: the deciding warp waiting for
// staged rows and in all; the feeder waiting for a free ring slot and for published summaries; the
// summary blocks waiting for published decisions, for probed rows, and evaluating rows; the probe
// blocks waiting for the inserts of earlier decisions.
enum : int {
  kGsFast = 0, kGsFull, kGsDecideWait, kGsDecideTotal, kGsFeedSlotWait, kGsFeedSumWait, kGsSumJobWait,
  kGsSumReadyWait, kGsSumEval, kGsProbeDoneWait, kGreedyStats
};

// Window table from a chain's last block hash to the earliest request ending there.
struct LastSlot {
  unsigned long long key;
  unsigned int neg_idx;  // 0xFFFFFFFF - request index (atomicMax keeps the earliest)
  unsigned int pad;
};

// Instance orders inside T (Table 4), as ps_model.selector.
enum : int32_t { kSelDCQ = 0, kSelD = 1, kSelDQ = 2, kSelDC = 3, kSelDQC = 4, kSelHCQ = 5 };

struct DevModel {
  float a0, a1, a2, a3, a4, a5, b0, b1, b2, g_q, eta, lout;
  int32_t interference_mode, ttft_filter, nseg;
  int32_t seg_lo[16];
  float ema[16];
  // policy variants of the evaluation (Table 3 admission ablations, Table 4 selectors); all zero is
  // Algorithm 1
  int32_t cache_off;  // 1: C = A (no KVC-first filter)
  int32_t slo_off;    // 1: T = C (no SLO admission)
  int32_t fb_dcq;     // 1: with T empty, the D-C-Q order over C instead of the LMetric product
  int32_t sel;        // order inside T (kSel*)
};

struct StateSoA {
  int32_t* b;
  int32_t* qr;
  int64_t* q;
  int64_t* S;
  int64_t* M;
  int32_t* Bmax;
};

struct WindowDev {
  const uint64_t* off;
  const uint64_t* hash;
  const uint32_t* L;
  const float* ttft_t;
  const float* tpot_t;
  uint32_t R;
};

__device__ __forceinline__ uint32_t fastrange32(uint64_t h, uint32_t n) {
  return (uint32_t)__umul64hi(h, (unsigned long long)n);
}

// Second bucket choice: an odd-constant multiply of a folded key, so fastrange of it uses bits
// independent of the ones that pick the first bucket.
__device__ __forceinline__ uint64_t remix(uint64_t k) { return (k ^ (k >> 31)) * 0x7FB5D329728EA185ull; }

// Membership in an instance's main table, in two parts so that several lookups can have their
// loads in flight together: lookup_issue requests both candidate buckets (2 x 4 x 16-byte loads)
// and the overflow word, lookup_finish compares (and, rarely, follows the overflow run after b1).
// RO selects the read path: the read-only path for kernels that never write the tables, the
// L2-coherent path for the table writers.
struct Lookup {
  ulonglong2 v[8];
  uint64_t ow;
  uint32_t b1;
};

template <bool RO = true>
__device__ __forceinline__ void lookup_issue(const uint64_t* __restrict__ slots, const uint64_t* __restrict__ ovf,
                                             const TableDesc& d, uint64_t key, Lookup& L) {
  L.b1 = fastrange32(key, d.nbkt);
  const uint32_t b2 = fastrange32(remix(key), d.nbkt);
  const ulonglong2* l1 = reinterpret_cast<const ulonglong2*>(slots + d.base + (uint64_t)L.b1 * kBucketSlots);
  const ulonglong2* l2 = reinterpret_cast<const ulonglong2*>(slots + d.base + (uint64_t)b2 * kBucketSlots);
#pragma unroll
  for (int k = 0; k < 4; ++k) {
    L.v[k] = RO ? __ldg(l1 + k) : __ldcg(l1 + k);
    L.v[4 + k] = RO ? __ldg(l2 + k) : __ldcg(l2 + k);
  }
  const uint64_t* ow_p = ovf + d.ovf + (L.b1 >> 6);
  L.ow = RO ? __ldg(ow_p) : __ldcg(ow_p);
}

template <bool RO = true>
__device__ __forceinline__ bool lookup_finish(const uint64_t* __restrict__ slots, const uint64_t* __restrict__ ovf,
                                              const TableDesc& d, uint64_t key, const Lookup& L) {
  if (key == kEmpty || key == kTomb) return false;
  bool hit = false;
#pragma unroll
  for (int k = 0; k < 8; ++k) hit |= (L.v[k].x == key) | (L.v[k].y == key);
  if (hit) return true;
  if (!((L.ow >> (L.b1 & 63)) & 1ull)) return false;
  uint32_t b = L.b1;  // rare: follow the overflow run after b1
  for (uint32_t p = 1; p < d.nbkt; ++p) {
    b = (b + 1 == d.nbkt) ? 0u : b + 1;
    const ulonglong2* l = reinterpret_cast<const ulonglong2*>(slots + d.base + (uint64_t)b * kBucketSlots);
#pragma unroll
    for (int k = 0; k < 4; ++k) {
      const ulonglong2 x = RO ? __ldg(l + k) : __ldcg(l + k);
      if (x.x == key || x.y == key) return true;
    }
    const uint64_t* q = ovf + d.ovf + (b >> 6);
    if (!(((RO ? __ldg(q) : __ldcg(q)) >> (b & 63)) & 1ull)) return false;
  }
  return false;
}

template <bool RO = true>
__device__ __forceinline__ bool main_contains(const uint64_t* __restrict__ slots, const uint64_t* __restrict__ ovf,
                                              const TableDesc d, uint64_t key) {
  if (key == kEmpty || key == kTomb) return false;
  Lookup L;
  lookup_issue<RO>(slots, ovf, d, key, L);
  return lookup_finish<RO>(slots, ovf, d, key, L);
}

// Global slot index of key in an instance's main table, or ~0 if absent (L2-coherent reads; used
// by the table writers).
__device__ __forceinline__ uint64_t main_find(const uint64_t* slots, const uint64_t* ovf, const TableDesc d,
                                              uint64_t key) {
  if (key == kEmpty || key == kTomb) return ~0ull;
  const uint32_t b1 = fastrange32(key, d.nbkt);
  const uint32_t b2 = fastrange32(remix(key), d.nbkt);
  const uint64_t s1 = d.base + (uint64_t)b1 * kBucketSlots, s2 = d.base + (uint64_t)b2 * kBucketSlots;
  ulonglong2 v[8];
#pragma unroll
  for (int k = 0; k < 4; ++k) {
    v[k] = __ldcg(reinterpret_cast<const ulonglong2*>(slots + s1) + k);
    v[4 + k] = __ldcg(reinterpret_cast<const ulonglong2*>(slots + s2) + k);
  }
  const uint64_t ow = __ldcg(ovf + d.ovf + (b1 >> 6));
#pragma unroll
  for (int k = 0; k < 4; ++k) {
    if (v[k].x == key) return s1 + 2 * k;
    if (v[k].y == key) return s1 + 2 * k + 1;
    if (v[4 + k].x == key) return s2 + 2 * k;
    if (v[4 + k].y == key) return s2 + 2 * k + 1;
  }
  if (!((ow >> (b1 & 63)) & 1ull)) return ~0ull;
  uint32_t b = b1;
  for (uint32_t p = 1; p < d.nbkt; ++p) {
    b = (b + 1 == d.nbkt) ? 0u : b + 1;
    const uint64_t sb = d.base + (uint64_t)b * kBucketSlots;
    for (int k = 0; k < kBucketSlots; ++k)
      if (__ldcg(reinterpret_cast<const unsigned long long*>(slots + sb + k)) == key) return sb + k;
    if (!((__ldcg(ovf + d.ovf + (b >> 6)) >> (b & 63)) & 1ull)) return ~0ull;
  }
  return ~0ull;
}

// Per-block LRU metadata, parallel to the slot array (streaming caches only): the block's last use,
// its number of cached children, and its parent's slot (kNoParent for a chain root or a parent that
// was not cached when the block was inserted).  A slot is stable while its block is cached and a
// parent outlives its children (eviction is leaf-first), so a cached block's parent slot stays valid.
constexpr uint64_t kNoParent = ~0ull;
constexpr uint64_t kLinkPending = ~1ull;  // inserted by a commit whose linking pass has not run yet
struct LruMeta {
  uint32_t* last_use;
  uint32_t* children;
  uint64_t* parent;
};

// Requests in flight per instance (streaming only): a FIFO ring of queued requests and an array of
// decoding ones, each of capacity M per instance.
struct ReqStore {
  uint32_t M;
  uint32_t* q_head;   // [I] ring start
  uint32_t* q_len;    // [I]
  uint32_t* q_L;      // [I*M]
  uint32_t* q_out;    // [I*M]
  uint64_t* q_rem;    // [I*M] remaining prefill tokens
  uint32_t* d_len;    // [I]
  uint32_t* d_L;      // [I*M]
  uint32_t* d_out;    // [I*M]
  uint32_t* d_rem;    // [I*M] remaining output tokens
};

// Warp-cooperative insert of one key by the instance's only writer warp (all 32 lanes call it with
// the same arguments).  Lanes 0-7 read bucket b1, lanes 8-15 bucket b2; the key goes to the emptier
// one.  With LRU metadata (meta.last_use != nullptr) a new block records (last_use, 0 children,
// its parent's slot) and its cached parent gains a child; an existing block only has its last_use
// raised.  parent_slot, if not ~0, is the parent's known slot (saves a lookup).  Returns the key's
// slot, or ~0 if the table is full; *inserted tells whether the key is new.
__device__ __forceinline__ uint64_t warp_insert(uint64_t* slots, uint64_t* ovf, const TableDesc d, uint64_t key,
                                                bool* inserted, LruMeta meta = LruMeta{nullptr, nullptr, nullptr},
                                                uint64_t parent = 0, uint32_t last_use = 0,
                                                uint64_t parent_slot = ~0ull) {
  const int lane = threadIdx.x & 31;
  *inserted = false;
  const uint64_t found = main_find(slots, ovf, d, key);
  if (found != ~0ull) {
    if (meta.last_use && lane == 0 && meta.last_use[found] < last_use) meta.last_use[found] = last_use;
    __syncwarp();
    return found;
  }
  const uint32_t b1 = fastrange32(key, d.nbkt);
  const uint32_t b2 = fastrange32(remix(key), d.nbkt);
  uint64_t idx = ~0ull;
  if (lane < 8) idx = d.base + (uint64_t)b1 * kBucketSlots + lane;
  else if (lane < 16) idx = d.base + (uint64_t)b2 * kBucketSlots + (lane - 8);
  const uint64_t v = idx != ~0ull ? __ldcg(reinterpret_cast<const unsigned long long*>(slots + idx)) : ~0ull;
  const unsigned empty = __ballot_sync(0xffffffffu, idx != ~0ull && v == kEmpty);
  const unsigned e1 = empty & 0xFFu, e2 = empty & 0xFF00u;
  int target = -1;
  if (e1 || e2) {
    // emptier bucket (more empty slots), b1 on ties
    target = (__popc(e1) >= __popc(e2)) ? __ffs(e1) - 1 : __ffs(e2) - 1;
  } else {
    // both full: first non-full bucket after b1; mark b1 and every full bucket passed
    uint32_t b = b1;
    for (uint32_t step = 0; step < d.nbkt && target < 0; ++step) {
      if (lane == 0) atomicOr(reinterpret_cast<unsigned long long*>(ovf + d.ovf + (b >> 6)), 1ull << (b & 63));
      b = (b + 1 == d.nbkt) ? 0u : b + 1;
      const uint64_t q = d.base + (uint64_t)b * kBucketSlots + (lane & 7);
      const uint64_t w = lane < 8 ? __ldcg(reinterpret_cast<const unsigned long long*>(slots + q)) : ~0ull;
      const unsigned em = __ballot_sync(0xffffffffu, lane < 8 && w == kEmpty);
      if (em) {
        target = __ffs(em) - 1;
        idx = q;
      }
    }
    if (target < 0) return ~0ull;
  }
  const uint64_t slot = __shfl_sync(0xffffffffu, idx, target);
  uint64_t ps = kNoParent;
  if (meta.last_use && parent != kEmpty) ps = parent_slot != ~0ull ? parent_slot : main_find(slots, ovf, d, parent);
  if (lane == target) {
    slots[slot] = key;
    if (meta.last_use) {
      meta.last_use[slot] = last_use;
      meta.children[slot] = 0;
      meta.parent[slot] = ps;
    }
  }
  if (ps != kNoParent && lane == 0) meta.children[ps] += 1;
  __syncwarp();
  *inserted = true;
  return slot;
}

// Insert of one key by one thread while other threads insert other keys into the same table (each
// key by one thread only; a key cached before the batch is found and left in place): both
// candidate buckets are read, the emptier one (b1 on ties) is tried first, a slot is claimed by
// compare-and-swap from empty, and if both buckets are full the key goes to the first bucket after
// b1 with a free slot, setting the overflow bit of b1 and of every full bucket passed (the layout
// lookups expect).  Placement can differ from a one-at-a-time build, the set of keys cannot.
// Returns the key's slot (~0: the table is full); *inserted tells whether this thread stored it.
__device__ __forceinline__ uint64_t thread_insert(uint64_t* slots, uint64_t* ovf, const TableDesc d, uint64_t key,
                                                  bool* inserted) {
  *inserted = false;
  const uint64_t found = main_find(slots, ovf, d, key);  // already cached before this batch of inserts
  if (found != ~0ull) return found;
  const uint32_t b1 = fastrange32(key, d.nbkt);
  const uint32_t b2 = fastrange32(remix(key), d.nbkt);
  auto try_bucket = [&](uint32_t b, uint64_t* out) -> int {  // 1 claimed, 0 full, -1 key found
    unsigned long long* base = reinterpret_cast<unsigned long long*>(slots + d.base + (uint64_t)b * kBucketSlots);
#pragma unroll 1
    for (int k = 0; k < kBucketSlots; ++k) {
      const unsigned long long v = __ldcg(base + k);
      if (v == key) {
        *out = d.base + (uint64_t)b * kBucketSlots + k;
        return -1;
      }
      if (v != kEmpty) continue;
      const unsigned long long old = atomicCAS(base + k, kEmpty, (unsigned long long)key);
      if (old == kEmpty || old == key) {
        *out = d.base + (uint64_t)b * kBucketSlots + k;
        return old == kEmpty ? 1 : -1;
      }
    }
    return 0;
  };
  auto empties = [&](uint32_t b) {
    const unsigned long long* base = reinterpret_cast<const unsigned long long*>(slots + d.base + (uint64_t)b * kBucketSlots);
    int n = 0;
#pragma unroll
    for (int k = 0; k < kBucketSlots; ++k) n += __ldcg(base + k) == kEmpty;
    return n;
  };
  uint64_t slot = ~0ull;
  const bool first_b1 = empties(b1) >= empties(b2);
  const uint32_t order[2] = {first_b1 ? b1 : b2, first_b1 ? b2 : b1};
  for (int c = 0; c < 2; ++c) {
    const int v = try_bucket(order[c], &slot);
    if (v != 0) {
      *inserted = v == 1;
      return slot;
    }
  }
  uint32_t b = b1;
  for (uint32_t step = 0; step < d.nbkt; ++step) {
    atomicOr(reinterpret_cast<unsigned long long*>(ovf + d.ovf + (b >> 6)), 1ull << (b & 63));
    b = (b + 1 == d.nbkt) ? 0u : b + 1;
    const int v = try_bucket(b, &slot);
    if (v != 0) {
      *inserted = v == 1;
      return slot;
    }
  }
  return ~0ull;
}

// The window's delta table: open addressing with linear probing over 16-byte slots, the home slot
// a function of the block hash alone, so lookups of one block for many instances read one line.
__device__ __forceinline__ uint64_t delta_home(uint64_t key, uint64_t nslots) { return __umul64hi(key, nslots); }

__device__ __forceinline__ uint64_t delta_next(uint64_t slot, uint64_t nslots) {
  return slot + 1 == nslots ? 0ull : slot + 1;
}

// Verdict of one slot for (key, tag = inst + 1): 1 present, 0 absent, -1 look at the next slot.
// Slots fill as an unbroken run from a key's home (inserts only claim empty slots and nothing is
// removed while a window runs), so an empty slot ends the search.  A slot of the key whose tag is
// not (yet) this instance's sends the search on: the pair is stored once, in its own slot.
__device__ __forceinline__ int delta_slot_verdict(const ulonglong2& v, uint64_t key, uint32_t tag) {
  if (v.x == key) return (uint32_t)v.y == tag ? 1 : -1;
  return v.x == kEmpty ? 0 : -1;
}

// Membership of (inst, key) from a given slot on, read through L2 (other blocks may be inserting).
__device__ __forceinline__ bool delta_contains_from(const DeltaSlot* delta, uint64_t nslots, uint32_t inst,
                                                    uint64_t key, uint64_t slot) {
  for (uint64_t p = 0; p < nslots; ++p) {
    const int v = delta_slot_verdict(__ldcg(reinterpret_cast<const ulonglong2*>(delta + slot)), key, inst + 1);
    if (v >= 0) return v == 1;
    slot = delta_next(slot, nslots);
  }
  return false;
}

__device__ __forceinline__ bool delta_contains(const DeltaSlot* delta, uint64_t nslots, uint32_t inst, uint64_t key) {
  if (key == kEmpty || key == kTomb) return false;
  return delta_contains_from(delta, nslots, inst, key, delta_home(key, nslots));
}

// Insert (inst, key) at the first empty slot from `slot` on (see delta_insert).
__device__ __forceinline__ bool delta_insert_from(DeltaSlot* delta, uint64_t nslots, uint32_t inst, uint64_t key,
                                                  uint64_t slot) {
  for (uint64_t p = 0; p < nslots; ++p) {
    if (atomicCAS(&delta[slot].hash, kEmpty, (unsigned long long)key) == kEmpty) {
      __stcg(&delta[slot].tag, inst + 1);
      return true;
    }
    slot = delta_next(slot, nslots);
  }
  return false;
}

// Insert (inst, key): the first empty slot from the key's home is claimed by compare-and-swap on
// the hash, then the tag is stored (one round trip).  A lookup racing with the insert may see the
// slot without its tag and report the pair absent, which only under-reports; it is visible to every
// reader once the inserting block has released its done flag.  The table has twice as many slots as
// a window has chain blocks, so it cannot fill; false reports a full table anyway.
__device__ __forceinline__ bool delta_insert(DeltaSlot* delta, uint64_t nslots, uint32_t inst, uint64_t key) {
  if (key == kEmpty || key == kTomb) return true;
  uint64_t slot = delta_home(key, nslots);
  for (uint64_t p = 0; p < nslots; ++p) {
    if (atomicCAS(&delta[slot].hash, kEmpty, (unsigned long long)key) == kEmpty) {
      __stcg(&delta[slot].tag, inst + 1);
      return true;
    }
    slot = delta_next(slot, nslots);
  }
  return false;
}

// ------------------------------------------------------------------ cross-block signalling (sm_90+) --
__device__ __forceinline__ uint32_t ld_acquire_u32(const uint32_t* p) {
  uint32_t v;
  asm volatile("ld.acquire.gpu.global.u32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
  return v;
}

__device__ __forceinline__ void st_release_u32(uint32_t* p, uint32_t v) {
  asm volatile("st.release.gpu.global.u32 [%0], %1;" ::"l"(p), "r"(v) : "memory");
}

__device__ __forceinline__ unsigned long long ld_relaxed_u64(const unsigned long long* p) {
  unsigned long long v;
  asm volatile("ld.relaxed.gpu.global.u64 %0, [%1];" : "=l"(v) : "l"(p) : "memory");
  return v;
}

__device__ __forceinline__ void st_relaxed_u64(unsigned long long* p, unsigned long long v) {
  asm volatile("st.relaxed.gpu.global.u64 [%0], %1;" ::"l"(p), "l"(v) : "memory");
}

// Shared-memory flags between the warps of one block: a release store at CTA scope (orders this
// thread's earlier accesses, without waiting for global stores).
__device__ __forceinline__ void st_release_cta_shared_u32(uint32_t* p, uint32_t v) {
  asm volatile("st.release.cta.shared::cta.u32 [%0], %1;" ::"r"((uint32_t)__cvta_generic_to_shared(p)), "r"(v)
               : "memory");
}

__device__ __forceinline__ uint32_t ld_relaxed_cta_shared_u32(const uint32_t* p) {
  uint32_t v;
  asm volatile("ld.relaxed.cta.shared::cta.u32 %0, [%1];" : "=r"(v) : "r"((uint32_t)__cvta_generic_to_shared(p))
               : "memory");
  return v;
}

// With a relaxed load before it that observed a release store, an acquire (CTA scope).
__device__ __forceinline__ void fence_acq_rel_cta() { asm volatile("fence.acq_rel.cta;" ::: "memory"); }

__device__ __forceinline__ uint64_t globaltimer_ns() {
  uint64_t x;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(x));
  return x;
}

// Bounded spin on a shared-memory counter until it reaches `want` (then an acquire fence) or *abort
// is set; false on timeout (error bit set) or abort.  An iteration is one shared load and a compare;
// the bound is counted in SM cycles, 3 per ns (at least the time limit at any clock up to 3 GHz).
__device__ __forceinline__ bool wait_smem_at_least(const uint32_t* p, uint32_t want, const volatile int* abort,
                                                   uint32_t* err, uint64_t limit_ns) {
  if (ld_relaxed_cta_shared_u32(p) >= want) {
    fence_acq_rel_cta();
    return true;
  }
  const long long c0 = clock64();
  const long long lim = (long long)(limit_ns * 3ull);
  for (uint32_t it = 1;; ++it) {
    if (ld_relaxed_cta_shared_u32(p) >= want) {
      fence_acq_rel_cta();
      return true;
    }
    if ((it & 31u) == 0u) {
      if (*abort) return false;
      if (clock64() - c0 > lim) {
        atomicOr(err, kErrTimeout);
        return false;
      }
    }
  }
}

// 16-byte asynchronous global -> shared copy (completes at cp_async_wait_all of the same thread).
__device__ __forceinline__ void cp_async16(void* smem, const void* gmem) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"((uint32_t)__cvta_generic_to_shared(smem)), "l"(gmem)
               : "memory");
}

__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }

__device__ __forceinline__ void cp_async_wait_all() { asm volatile("cp.async.wait_all;" ::: "memory"); }

// ------------------------------------------------------------------------------- first-miss walks --
// All 32 lanes of a warp call these with the same arguments; present(k) is evaluated per lane.
// Each returns the first position k in [lo, nb) with present(k) false (nb if there is none), given
// that every position below lo is known present.

// Linear walk, 32 consecutive positions per step: exact for any membership pattern.
template <class Pred>
__device__ __forceinline__ uint64_t warp_first_miss_linear(uint64_t lo, uint64_t nb, Pred present) {
  const int lane = threadIdx.x & 31;
  for (uint64_t base = lo; base < nb; base += 32) {
    const uint64_t k = base + lane;
    const bool p = k < nb ? present(k) : true;
    const unsigned miss = __ballot_sync(0xffffffffu, !p);
    if (miss) return base + (uint64_t)(__ffs(miss) - 1);
  }
  return nb;
}

// 32-ary search, exact when membership is monotone along the chain (a prefix-closed cache).
// Invariant: the answer h lies in [lo, hi], positions below lo are present and position hi is
// absent (or hi = nb).  Each step probes 32 evenly spaced positions p_j = lo + (j+1) span / 32 - 1
// (p_31 = hi - 1) and keeps [p_{j-1} + 1, p_j] around the first miss j, so an interval of span s
// shrinks to at most ceil(s / 32); spans <= 32 are finished by one linear step.
template <class Pred>
__device__ __forceinline__ uint64_t warp_search_range(uint64_t lo, uint64_t hi, Pred present) {
  const int lane = threadIdx.x & 31;
  for (;;) {
    const uint64_t span = hi - lo;
    if (span == 0) return lo;
    if (span <= 32) {
      const uint64_t k = lo + lane;
      const bool p = k < hi ? present(k) : true;
      const unsigned miss = __ballot_sync(0xffffffffu, !p);
      return miss ? lo + (uint64_t)(__ffs(miss) - 1) : hi;
    }
    const uint64_t k = lo + ((uint64_t)(lane + 1) * span) / 32 - 1;
    const unsigned miss = __ballot_sync(0xffffffffu, !present(k));
    if (!miss) return hi;
    const uint64_t j = (uint64_t)(__ffs(miss) - 1);
    const uint64_t pj = lo + ((j + 1) * span) / 32 - 1;
    lo = lo + (j * span) / 32;
    hi = pj;
  }
}

__device__ __forceinline__ uint64_t warp_min_u64(uint64_t x) {
#pragma unroll
  for (int s = 16; s > 0; s >>= 1) {
    const uint64_t o = __shfl_xor_sync(0xffffffffu, x, s);
    x = o < x ? o : x;
  }
  return x;
}

__device__ __forceinline__ uint64_t warp_max_u64(uint64_t x) {
#pragma unroll
  for (int s = 16; s > 0; s >>= 1) {
    const uint64_t o = __shfl_xor_sync(0xffffffffu, x, s);
    x = o > x ? o : x;
  }
  return x;
}

// The same search with a likely answer (positions below lo are known present, lo itself need not
// be): the first step probes hint - 1 and hint next to 30 evenly spaced positions.  Under monotone membership every probed position narrows the interval (a
// present p raises lo to p + 1, an absent p lowers hi to p), so any positions keep it exact; when
// the hint is the answer the first step ends the search.
template <class Pred>
__device__ __forceinline__ uint64_t warp_first_miss_search_hint(uint64_t lo, uint64_t nb, uint64_t hint,
                                                                Pred present) {
  const int lane = threadIdx.x & 31;
  const uint64_t span = nb - lo;
  if (span <= 32 || hint <= lo || hint > nb) return warp_search_range(lo, nb, present);
  uint64_t p;
  if (lane == 0) p = hint - 1;
  else if (lane == 1) p = hint < nb ? hint : hint - 1;
  else p = lo + ((uint64_t)(lane - 1) * span) / 31 - 1;
  const bool pr = present(p);
  const uint64_t new_hi = warp_min_u64(pr ? ~0ull : p);
  const uint64_t last_present = warp_max_u64(pr ? p + 1 : 0ull);
  const uint64_t hi = new_hi == ~0ull ? nb : new_hi;
  uint64_t lo2 = last_present > lo ? last_present : lo;
  // A table read while inserts land need not look monotone: a present position may lie above an
  // absent one.  Every present answer is cached in the final set and every absent answer is not
  // cached in the set the inserts started from, so any point between them keeps the result between
  // the two sets' first misses; clamping also keeps the remaining range well formed.
  if (lo2 > hi) lo2 = hi;
  return warp_search_range(lo2, hi, present);
}

// ---------------------------------------------------------------------------- performance model --
// Every operation is an explicitly rounded fp32 intrinsic in the order the header documents, so
// nothing is fused or reassociated.

// int64 -> fp32, round to nearest: the 32-bit conversion when the value fits (the same result).  The
// 64-bit conversion is kept out of line, so values that fit (all token counts here) never issue it.
static __device__ __noinline__ float i64_to_f32_wide(int64_t v) { return __ll2float_rn(v); }
__device__ __forceinline__ float i64_to_f32(int64_t v) {
  if (v == (int64_t)(int32_t)v) return __int2float_rn((int32_t)v);
  return i64_to_f32_wide(v);
}

// Eq. 6 with the Section 5.3 empirical C and C^2 terms.
__device__ __forceinline__ float t_pf(const DevModel& m, float N, float C) {
  float t = __fadd_rn(m.a0, __fmul_rn(m.a1, N));
  t = __fadd_rn(t, __fmul_rn(m.a2, __fmul_rn(N, C)));
  t = __fadd_rn(t, __fmul_rn(m.a3, __fmul_rn(N, N)));
  t = __fadd_rn(t, __fmul_rn(m.a4, C));
  t = __fadd_rn(t, __fmul_rn(m.a5, __fmul_rn(C, C)));
  return t;
}

// Per-request constants of Algorithm 1 and Eq. 8.
struct RowConst {
  float t_cached;     // T_pf(0, L): fully cached input
  float Z;            // CacheBenefit: T_pf(L, 0) - T_pf(0, L)
  float etaZ;         // eta * Z
  float ttft_budget;  // max(target, T_pf(L, 0))
  float tpot_target;
  uint32_t L;
};

// Z of a row as the recompute filter uses it: without the KVC-first filter (Table 3) every pair of A
// is in C, which the filter's own rule gives for Z <= 0.
__device__ __forceinline__ float filter_z(const DevModel& m, float Z) { return m.cache_off ? 0.0f : Z; }

__device__ __forceinline__ RowConst row_const(const DevModel& m, uint32_t L, float ttft_t, float tpot_t) {
  RowConst rc;
  const float Lf = __uint2float_rn(L);
  rc.t_cached = t_pf(m, 0.0f, Lf);
  const float t_cold = t_pf(m, Lf, 0.0f);
  rc.Z = filter_z(m, __fsub_rn(t_cold, rc.t_cached));
  rc.etaZ = __fmul_rn(m.eta, rc.Z);
  rc.ttft_budget = t_cold > ttft_t ? t_cold : ttft_t;
  rc.tpot_target = tpot_t;
  rc.L = L;
  return rc;
}

struct PairEval {
  float W, tpot, ttft;
  int64_t n;   // uncached tokens
  bool inA;    // capacity-eligible
};

__device__ __forceinline__ float ema_factor(const DevModel& m, int64_t B) {
  if (m.nseg == 1) return m.ema[0];
  int s = 0;
  for (int k = 0; k < m.nseg; ++k)
    if ((int64_t)m.seg_lo[k] <= B) s = k;
  return m.ema[s];
}

// RecomputeCost, capacity guard and the latency predictions of one (request, instance) pair.
__device__ __forceinline__ PairEval eval_pair(const DevModel& m, const RowConst& rc, uint32_t h,
                                              int32_t b, int32_t qr, int64_t q, int64_t S, int64_t M,
                                              int32_t Bmax) {
  PairEval e;
  const int64_t c = 16 * (int64_t)h;
  const int64_t n = (int64_t)rc.L - c;
  const float tpf = t_pf(m, i64_to_f32(n), i64_to_f32(c));
  e.n = n;
  e.W = __fsub_rn(tpf, rc.t_cached);
  const int64_t Bp = (int64_t)b + qr + 1;
  const int64_t Sp = S + (int64_t)rc.L;
  e.inA = (Bp <= (int64_t)Bmax) && (Sp <= M);
  float dec = __fadd_rn(m.b0, __fmul_rn(m.b1, i64_to_f32(Bp)));
  dec = __fadd_rn(dec, __fmul_rn(m.b2, i64_to_f32(Sp)));
  dec = __fmul_rn(dec, ema_factor(m, Bp));
  if (m.interference_mode == 0) {
    e.tpot = __fadd_rn(dec, __fmul_rn(m.g_q, i64_to_f32(q + n)));
  } else {
    const float den = m.lout > 1.0f ? m.lout : 1.0f;
    const float interf = ((int64_t)b + qr > 0) ? __fdiv_rn(tpf, den) : 0.0f;
    e.tpot = __fadd_rn(dec, interf);
  }
  const float tq = __fadd_rn(__fmul_rn(m.a0, __int2float_rn(qr)), __fmul_rn(m.a1, i64_to_f32(q)));
  e.ttft = __fadd_rn(tpf, tq);
  return e;
}

// Terms of eval_pair that depend only on the instance state (b, qr, q, B_max): they change only
// when the instance is picked, so the greedy keeps them per instance.  Same rounded operations as
// eval_pair, so results are bit-identical.
struct InstTerms {
  float dec0;   // b0 + b1 * B, B = b + qr + 1
  float f;      // EMA factor of B's segment
  float tq;     // a0 * qr + a1 * q (queueing part of TTFT)
  int32_t Bp;   // b + qr + 1
  int32_t okB;  // B <= B_max
};

// Free KV room M_KV - S of an instance clamped to [-1, 2^31 - 1]: for 0 <= L < 2^30 the capacity
// test S + L <= M_KV is L <= room.
__device__ __forceinline__ int32_t kv_room(int64_t S, int64_t M) {
  const int64_t d = M - S;
  return d < 0 ? -1 : (d > 0x7FFFFFFFll ? 0x7FFFFFFF : (int32_t)d);
}

__device__ __forceinline__ InstTerms inst_terms(const DevModel& m, int32_t b, int32_t qr, int64_t q, int32_t Bmax) {
  InstTerms x;
  const int64_t Bp = (int64_t)b + qr + 1;
  x.dec0 = __fadd_rn(m.b0, __fmul_rn(m.b1, i64_to_f32(Bp)));
  x.f = ema_factor(m, Bp);
  x.tq = __fadd_rn(__fmul_rn(m.a0, __int2float_rn(qr)), __fmul_rn(m.a1, i64_to_f32(q)));
  x.Bp = (int32_t)Bp;
  x.okB = Bp <= (int64_t)Bmax;
  return x;
}

// T_pf of a pair from its hit h: n = L - 16 h uncached tokens, c = 16 h cached.
__device__ __forceinline__ float t_pf_of_hit(const DevModel& m, uint32_t L, uint32_t h) {
  const int64_t c = 16 * (int64_t)h;
  return t_pf(m, i64_to_f32((int64_t)L - c), i64_to_f32(c));
}

// T_pf at hit h of a request of L tokens, in 32-bit integers: c = 16 h and n = L - c are below 2^30
// in magnitude (L < 2^30, h <= L / 16), so their conversions equal the 64-bit ones.
__device__ __forceinline__ float t_pf32(const DevModel& m, uint32_t L, uint32_t h) {
  const int32_t c = (int32_t)(h << 4);
  return t_pf(m, __int2float_rn((int32_t)L - c), __int2float_rn(c));
}

// TPOT and TTFT of a pair (pair_lat's rounded operations) with S + L and q + n formed in 32 bits, for
// instances whose q and S lie in [0, 2^30) (n = L - 16 h, L < 2^30).
__device__ __forceinline__ void pair_lat32(const DevModel& m, const RowConst& rc, float tpf, int32_t n, float dec0,
                                           float f, float tq, int32_t Bp, int32_t q32, int32_t S32, float* tpot,
                                           float* ttft) {
  float dec = __fadd_rn(dec0, __fmul_rn(m.b2, __int2float_rn(S32 + (int32_t)rc.L)));
  dec = __fmul_rn(dec, f);
  if (m.interference_mode == 0) {
    *tpot = __fadd_rn(dec, __fmul_rn(m.g_q, __int2float_rn(q32 + n)));
  } else {
    const float den = m.lout > 1.0f ? m.lout : 1.0f;
    *tpot = __fadd_rn(dec, Bp > 1 ? __fdiv_rn(tpf, den) : 0.0f);
  }
  *ttft = __fadd_rn(tpf, tq);
}

// Marks a precomputed T_pf as not available (a NaN pattern T_pf never produces).
constexpr uint32_t kNoTpfBits = 0xFFFFFFFFu;

// The two halves of eval_pair with the instance terms precomputed (the greedy evaluates the
// latencies only for pairs that pass the capacity guard and the recompute filter).  Together they
// perform exactly eval_pair's rounded operations.
//   pair_w:   T_pf at the hit (given unless tpf_in carries kNoTpfBits), W = T_pf(n, c) - T_pf(0, L),
//             n, and the capacity guard (Algorithm 1 CapacityCandidates).
//   pair_lat: TPOT (Eq. 5 / Eq. 9) and TTFT (Eq. 4) of the pair.
struct PairW {
  float W, tpf;
  int64_t n;
  bool inA;
};

__device__ __forceinline__ PairW pair_w(const DevModel& m, const RowConst& rc, uint32_t h, float tpf_in,
                                        const InstTerms& it, int64_t S, int64_t M) {
  PairW x;
  const int64_t c = 16 * (int64_t)h;
  x.n = (int64_t)rc.L - c;
  x.tpf = __float_as_uint(tpf_in) == kNoTpfBits ? t_pf(m, i64_to_f32(x.n), i64_to_f32(c)) : tpf_in;
  x.W = __fsub_rn(x.tpf, rc.t_cached);
  x.inA = it.okB && (S + (int64_t)rc.L <= M);
  return x;
}

__device__ __forceinline__ void pair_lat(const DevModel& m, const RowConst& rc, const PairW& x, const InstTerms& it,
                                         int64_t q, int64_t S, float* tpot, float* ttft) {
  const int64_t Sp = S + (int64_t)rc.L;
  float dec = __fadd_rn(it.dec0, __fmul_rn(m.b2, i64_to_f32(Sp)));
  dec = __fmul_rn(dec, it.f);
  if (m.interference_mode == 0) {
    *tpot = __fadd_rn(dec, __fmul_rn(m.g_q, i64_to_f32(q + x.n)));
  } else {
    const float den = m.lout > 1.0f ? m.lout : 1.0f;
    const float interf = (it.Bp > 1) ? __fdiv_rn(x.tpf, den) : 0.0f;
    *tpot = __fadd_rn(dec, interf);
  }
  *ttft = __fadd_rn(x.tpf, it.tq);
}

// eval_pair with the instance terms precomputed, and T_pf given unless it carries kNoTpfBits.
__device__ __forceinline__ PairEval eval_pair_tpf(const DevModel& m, const RowConst& rc, uint32_t h, float tpf_in,
                                                  const InstTerms& it, int64_t q, int64_t S, int64_t M) {
  const PairW x = pair_w(m, rc, h, tpf_in, it, S, M);
  PairEval e;
  e.n = x.n;
  e.W = x.W;
  e.inA = x.inA;
  pair_lat(m, rc, x, it, q, S, &e.tpot, &e.ttft);
  return e;
}

// Recompute filter (Eq. 8) of a capacity-eligible pair once W_min is known: W - W_min <= eta Z,
// every pair of A when Z <= 0.
__device__ __forceinline__ bool pair_in_c(const RowConst& rc, float W, float Wmin) {
  return (rc.Z > 0.0f) ? (__fsub_rn(W, Wmin) <= rc.etaZ) : true;
}

// Admission of a pair of C (Algorithm 1 TPOT filter, plus the TTFT budget when enabled; every pair
// of C without the SLO admission, Table 3).
__device__ __forceinline__ bool pair_admitted(const DevModel& m, const RowConst& rc, float tpot, float ttft) {
  if (m.slo_off) return true;
  bool ok = tpot < rc.tpot_target;
  if (m.ttft_filter) ok = ok && (ttft <= rc.ttft_budget);
  return ok;
}

__device__ __forceinline__ PairEval eval_pair_terms(const DevModel& m, const RowConst& rc, uint32_t h,
                                                    const InstTerms& it, int64_t q, int64_t S, int64_t M) {
  return eval_pair_tpf(m, rc, h, __uint_as_float(kNoTpfBits), it, q, S, M);
}

// Class of a capacity-eligible pair once W_min is known (Eq. 8, Alg. 1 TPOT filter + TTFT budget):
// 0 in T, 1 in C \ T, 2 filtered by the recompute budget.
__device__ __forceinline__ uint32_t pair_class(const DevModel& m, const RowConst& rc, const PairEval& e,
                                               float Wmin) {
  if (!pair_in_c(rc, e.W, Wmin)) return 2u;
  return pair_admitted(m, rc, e.tpot, e.ttft) ? 0u : 1u;
}

// Order-preserving map of a non-NaN float to an unsigned integer (for integer warp reductions).
__device__ __forceinline__ uint32_t f2ord(float x) {
  const uint32_t u = __float_as_uint(x);
  return (u & 0x80000000u) ? ~u : (u | 0x80000000u);
}
__device__ __forceinline__ float ord2f(uint32_t o) {
  return __uint_as_float((o & 0x80000000u) ? (o & 0x7FFFFFFFu) : ~o);
}

// ---- packing keys under the policy variants ---------------------------------------------------
// Class-0 value fields: D = 2^18-1-b (18 bits), C = 2^26-1-h (26 bits), Q = qr (18 bits), so a
// smaller value means more decoding requests, more cached blocks, fewer queued requests.
//   D-C-Q  D << 44 | C << 18 | Q        D    D << 44             D-Q  D << 44 | Q
//   D-C    D << 44 | C << 18            D-Q-C  D << 44 | Q << 26 | C
//   H-C-Q  ord(tpot_target - TPOT) << 26 | C, with Q carried in the tie word (qr << 12 | instance)
// The instance-only fields (D, Q) are kept per instance (key0_bits); a pair adds its hit field.
__device__ __forceinline__ uint64_t dcq_key0(int32_t b, int32_t qr) {
  return ((uint64_t)((1u << 18) - 1u - (uint32_t)b) << 44) | (uint64_t)(uint32_t)qr;
}

__device__ __forceinline__ uint64_t key0_bits(const DevModel& m, int32_t b, int32_t qr) {
  const uint64_t D = (uint64_t)((1u << 18) - 1u - (uint32_t)b) << 44;
  switch (m.sel) {
    case kSelDCQ:
    case kSelDQ: return D | (uint64_t)(uint32_t)qr;
    case kSelDQC: return D | ((uint64_t)(uint32_t)qr << 26);
    case kSelHCQ: return 0ull;
    default: return D;
  }
}

__device__ __forceinline__ uint64_t hit_bits(const DevModel& m, uint32_t h) {
  const uint64_t C = (uint64_t)((1u << 26) - 1u - h);
  if (m.sel == kSelDCQ || m.sel == kSelDC) return C << 18;
  if (m.sel == kSelDQC || m.sel == kSelHCQ) return C;
  return 0ull;
}

// key0_bits from the D-C-Q bits of (b, qr) (dcq_key0), which is what kernels keep per instance.
__device__ __forceinline__ uint64_t key0_from_dcq(const DevModel& m, uint64_t kd) {
  if (m.sel == kSelDCQ) return kd;
  return key0_bits(m, (int32_t)((1u << 18) - 1u - (uint32_t)(kd >> 44)), (int32_t)(kd & 0x3FFFFull));
}

// Value of a pair of T (class 0) from its instance's key0_bits, hit and predicted TPOT.
__device__ __forceinline__ uint64_t value_in_t(const DevModel& m, uint64_t k0, uint32_t h, float tpot, float target) {
  uint64_t v = k0 | hit_bits(m, h);
  if (m.sel == kSelHCQ) v |= (uint64_t)f2ord(__fsub_rn(target, tpot)) << 26;
  return v;
}

// Tie word of a pair of T: the instance id, or qr << 12 | id under H-C-Q (ids < 4096).
__device__ __forceinline__ uint32_t tie_in_t(const DevModel& m, uint32_t i, int32_t qr) {
  return m.sel == kSelHCQ ? (((uint32_t)qr << 12) | i) : i;
}
constexpr uint32_t kTieInstMask = 0xFFFu;

// Value of a pair of C \ T (class 1): the LMetric product (q + n)(b + qr + 1), or the D-C-Q value
// under the ablations' D-C-Q fallback (kd = dcq_key0(b, qr)).
__device__ __forceinline__ uint64_t value_fallback(const DevModel& m, uint64_t qn, uint32_t Bp, uint64_t kd,
                                                   uint32_t h) {
  if (m.fb_dcq) return kd | ((uint64_t)((1u << 26) - 1u - h) << 18);
  return qn * (uint64_t)Bp;
}

__device__ __forceinline__ float warp_fmin(float x) {
#pragma unroll
  for (int s = 16; s > 0; s >>= 1) x = fminf(x, __shfl_xor_sync(0xffffffffu, x, s));
  return x;
}

// (class, value) of a pair of C as one 64-bit key, class in the top two bits: class-0 values are
// below 2^62 and class-1 values below 2^59 ((q + n) < 2^41 times (b + qr + 1) < 2^18), so the
// unsigned order of the packed key is the lexicographic order of (class, value).
__device__ __forceinline__ uint64_t packed_key(uint32_t cls, uint64_t v) { return ((uint64_t)cls << 62) | v; }
constexpr uint64_t kNoKey = ~0ull;

// Warp argmin of (key, instance) with single-instruction reductions; every lane receives the
// minimum and the winning lane's h.  Lanes without a pair pass (kNoKey, 0xFFFFFFFF).
__device__ __forceinline__ void warp_pick_min(uint64_t key, uint32_t inst, uint32_t h, uint64_t* kout,
                                              uint32_t* iout, uint32_t* hout) {
  const uint32_t hi = (uint32_t)(key >> 32);
  const uint32_t mhi = __reduce_min_sync(0xffffffffu, hi);
  const uint32_t lo = hi == mhi ? (uint32_t)key : 0xFFFFFFFFu;
  const uint32_t mlo = __reduce_min_sync(0xffffffffu, lo);
  const bool eq = hi == mhi && (uint32_t)key == mlo;
  const uint32_t mi = __reduce_min_sync(0xffffffffu, eq ? inst : 0xFFFFFFFFu);
  const unsigned win = __ballot_sync(0xffffffffu, eq && inst == mi);
  *hout = __shfl_sync(0xffffffffu, h, __ffs(win) - 1);
  *kout = ((uint64_t)mhi << 32) | mlo;
  *iout = mi;
}

}  // namespace psk

namespace psk {
// Scoring over one column block of an instance pool (the pool's instances split over contexts, one
// block each).  Algorithm 1 is a map over instances followed by two reductions per request: W_min
// over A, then the smallest (key, tie) over C.  A block's kernel computes its part of each, and the
// caller combines them across blocks (a MIN over blocks):
//   wmin_out  non-null: write the block's W_min over A (f2ord bits, 0xFFFFFFFF = A empty) per request
//             and stop after it (no classes, latencies or pick);
//   wmin_in   non-null: use the pool's W_min (f2ord bits, per request) in the recompute filter instead
//             of the block's own;
//   key_out, tie_out  non-null: the block's smallest packed key per request (kNoKey if none) and its
//             tie word with the pool's instance id (id_base + local id; under H-C-Q qr << 12 | id).
struct ShardIO {
  const uint32_t* wmin_in = nullptr;
  uint32_t* wmin_out = nullptr;
  unsigned long long* key_out = nullptr;
  uint32_t* tie_out = nullptr;
  uint32_t id_base = 0;
};
}  // namespace psk

// Kernel launchers (one translation unit each).
namespace pskl {
// rows (from launch_relations, or nullptr to probe every request from scratch); tpf (nullable)
// receives T_pf of every pair's hit; stats (nullable) accumulates the six launch counters of
// ps_last_probe_stats; ev_mid (nullable) is recorded between the two probe kernels.
cudaError_t launch_probe(const uint64_t* slots, const uint64_t* ovf, const psk::TableDesc* tdesc, uint32_t I,
                         const psk::WindowDev& w, const psk::RowPre* rows, psk::RowList list, uint32_t* hits,
                         float* tpf, const psk::DevModel& m, int grid, int search, unsigned long long* stats,
                         cudaEvent_t ev_mid, cudaStream_t s);
int probe_max_grid(uint32_t I, int num_sms);
cudaError_t launch_score(const uint32_t* hits, psk::StateSoA st, uint32_t I, const psk::WindowDev& w,
                         const psk::DevModel& m, float* tpot, float* ttft, uint8_t* cls, int32_t* best,
                         uint8_t* path, int num_sms, cudaStream_t s, const psk::ShardIO& sh = psk::ShardIO());
cudaError_t launch_greedy(const uint64_t* slots, const uint64_t* ovf, const psk::TableDesc* tdesc, uint32_t I,
                          const psk::WindowDev& w, const uint32_t* hit0, psk::StateSoA committed,
                          psk::StateSoA pending, const psk::DevModel& m, psk::DeltaSlot* delta,
                          uint64_t delta_nslots, int32_t* assign, uint8_t* path, uint32_t* hit_chosen,
                          uint32_t* err, int search, cudaStream_t s);
cudaError_t launch_delta_clear(psk::DeltaSlot* delta, uint64_t nslots, cudaStream_t s);
// Rebuilds every chain of a window in the shared-prefix form (ps_window.parent) into hash (CSR at
// full_off) from each request's own blocks (CSR at own_off) and its parent link.
cudaError_t launch_expand_chains(const uint64_t* full_off, const uint64_t* own_off, const uint64_t* own_hash,
                                 const int32_t* parent, uint32_t R, uint64_t* hash, uint32_t* err, int num_sms,
                                 cudaStream_t s);
cudaError_t launch_relations(const psk::WindowDev& w, const psk::DevModel& m, psk::LastSlot* tab, uint32_t tab_n,
                             psk::RowPre* rows, psk::RowList list, int num_sms, cudaStream_t s);
cudaError_t launch_greedy_search(const psk::RowPre* rows, const psk::WindowDev& w, uint32_t I, const uint32_t* hit0,
                                 const float* tpf0, psk::StateSoA committed, psk::StateSoA pending, const psk::DevModel& m,
                                 psk::DeltaSlot* delta, uint64_t delta_nslots, int32_t* assign, uint8_t* path,
                                 uint32_t* hit_chosen, uint32_t* err, const psk::GreedySync& sync, cudaStream_t s);
cudaError_t launch_insert_chains(uint64_t* slots, uint64_t* ovf, const psk::TableDesc* tdesc, uint32_t I,
                                 unsigned long long* count, uint64_t nchains, const uint32_t* inst,
                                 const uint64_t* off, const uint64_t* hash, const uint64_t* parent,
                                 uint64_t total, psk::LruMeta meta, uint32_t last_use, uint32_t* err,
                                 int num_sms, cudaStream_t s);
// prefix: device scratch of 2 (R + 1) words.
cudaError_t launch_commit(uint64_t* slots, uint64_t* ovf, const psk::TableDesc* tdesc, uint32_t I,
                          unsigned long long* count, const psk::WindowDev& w, const int32_t* assign,
                          const uint32_t* hit_chosen, psk::LruMeta meta, uint32_t last_use,
                          const psk::ReqStore& rq, const uint32_t* out_tokens, unsigned long long* prefix,
                          uint32_t* err, int num_sms, cudaStream_t s);
cudaError_t launch_advance(psk::StateSoA st, uint32_t I, const psk::ReqStore& rq, const psk::DevModel& m,
                           float window_ms, uint64_t prefill_tokens, uint32_t* err, cudaStream_t s);
// Leaf-first LRU eviction of every instance over capacity (rounds until none is; synchronises the
// stream between rounds).  leafbuf holds evict_leafbuf_bytes(I) bytes; nleaf [I], more [1] device
// words; more_host one pinned word; max_instance_slots the largest table (slots) of an instance.
cudaError_t launch_evict(uint64_t* slots, const psk::TableDesc* tdesc, uint32_t I, unsigned long long* count,
                         const uint64_t* cap, psk::LruMeta meta, void* leafbuf, uint32_t* nleaf, uint32_t* more,
                         uint32_t* more_host, uint64_t max_instance_slots, uint32_t* err, cudaStream_t s);
size_t evict_leafbuf_bytes(uint32_t I);
cudaError_t launch_check_parents(const uint64_t* slots, const uint64_t* ovf, const psk::TableDesc* tdesc, uint32_t I,
                                 uint64_t nchains, const uint32_t* inst, const uint64_t* parent,
                                 uint32_t* err, int num_sms, cudaStream_t s);
cudaError_t launch_validate_window(const psk::WindowDev& w, uint64_t max_blocks, uint32_t* err,
                                   cudaStream_t s);
}  // namespace pskl
