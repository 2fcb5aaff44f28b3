// Fused score kernel: hit lengths + instance state -> predicted latencies, Algorithm 1's admission
// sets and the per-request pick, each request independently against the same state.
//
// Two forms: score_block_kernel for rows of 257 .. 1024 instances (a thread block per row, the
// instance terms in registers; described at its section below) and score_rows_kernel for the other
// sizes, described here.  The instance terms that do not depend on the request (InstTerms, the free KV room with the
// decode-slot guard folded in, q, S and the class-0 key bits of (b, qr)) are computed once per
// thread block into shared memory as padded structure-of-arrays.  One warp then takes one request
// at a time: lane l owns the instances 128 v + 4 l .. 128 v + 4 l + 3 of each 128-instance chunk v,
// so a row of hits is read with one 16-byte load per lane and chunk, and the per-pair outputs
// (TPOT, TTFT as float4, the classes as one 32-bit word) are written with one store per lane and
// chunk.  Pass 1 evaluates the capacity guard and the recompute cost W (Alg. 1 KVC-first filtering)
// and reduces W_min over A; pass 2 classifies each pair (Eq. 8 filter, TPOT and TTFT admission)
// and reduces the packed (class, value) key to the pick: D-C-Q inside T, the LMetric product inside
// C when T is empty, Reject when A is empty (or the model's policy variant of Table 3 / Table 4).
// Pass 2 takes the hits from registers; rows of more than 128 NV instances are taken in pieces of
// NV chunks, each read again for pass 2.
#include <type_traits>

#include "ps_internal.cuh"

namespace {

constexpr int kScoreThreads = 256;

// Shared-memory instance arrays, each [Ip] (I rounded up to a multiple of 4), 8-byte arrays first.
// q32 / S32 are 32-bit copies of q / S, used when every instance of the block has both in
// [0, 2^30): then S + L and q + n (L, n < 2^30) are exact in 32 bits.
struct ScoreSmem {
  int64_t* q;
  int64_t* S;
  uint64_t* k0;    // D-C-Q key bits of (b, qr) (psk::dcq_key0; other orders derive theirs)
  int32_t* room;   // free KV room M_KV - S, -1 when the decode-slot guard fails or past I
  float* dec0;
  float* f;
  float* tq;
  int32_t* Bp;
  int32_t* q32;
  int32_t* S32;
};

__device__ __forceinline__ ScoreSmem score_smem(unsigned long long* raw, uint32_t Ip) {
  ScoreSmem s;
  s.q = reinterpret_cast<int64_t*>(raw);
  s.S = s.q + Ip;
  s.k0 = reinterpret_cast<uint64_t*>(s.S + Ip);
  s.room = reinterpret_cast<int32_t*>(s.k0 + Ip);
  s.dec0 = reinterpret_cast<float*>(s.room + Ip);
  s.f = s.dec0 + Ip;
  s.tq = s.f + Ip;
  s.Bp = reinterpret_cast<int32_t*>(s.tq + Ip);
  s.q32 = s.Bp + Ip;
  s.S32 = s.q32 + Ip;
  return s;
}

// Four consecutive shared-memory elements (16-byte aligned) with 16-byte loads.
__device__ __forceinline__ void lds4(const float* p, float (&v)[4]) {
  const float4 x = *reinterpret_cast<const float4*>(p);
  v[0] = x.x;
  v[1] = x.y;
  v[2] = x.z;
  v[3] = x.w;
}
__device__ __forceinline__ void lds4(const int32_t* p, int32_t (&v)[4]) {
  const int4 x = *reinterpret_cast<const int4*>(p);
  v[0] = x.x;
  v[1] = x.y;
  v[2] = x.z;
  v[3] = x.w;
}
__device__ __forceinline__ void lds4(const int64_t* p, int64_t (&v)[4]) {
  const longlong2 x = reinterpret_cast<const longlong2*>(p)[0];
  const longlong2 y = reinterpret_cast<const longlong2*>(p)[1];
  v[0] = x.x;
  v[1] = x.y;
  v[2] = y.x;
  v[3] = y.y;
}
__device__ __forceinline__ void lds4(const uint64_t* p, uint64_t (&v)[4]) {
  const ulonglong2 x = reinterpret_cast<const ulonglong2*>(p)[0];
  const ulonglong2 y = reinterpret_cast<const ulonglong2*>(p)[1];
  v[0] = x.x;
  v[1] = x.y;
  v[2] = y.x;
  v[3] = y.y;
}

using psk::pair_lat32;
using psk::t_pf32;

// One piece of a row: NV chunks of 128 instances starting at instance i_lo.
template <int NV>
struct Piece {
  uint32_t h[NV][4];
  uint32_t amask;  // bit 4 v + k: the pair is in A
};

// Loads a piece's hits and evaluates pass 1: the capacity guard and, for pairs in A, T_pf at the hit
// and W = T_pf(n, c) - T_pf(0, L).  Returns the order-preserving bits of the lane's W_min over A
// (all ones if none).  With a stash (this warp's [Ip] scratch row in shared memory) T_pf of every
// pair pass 2 will need (all pairs when every per-pair output is wanted, else the pairs in A) is
// kept there, so pass 2 reads it instead of evaluating it again.
template <int NV, bool VEC>
__device__ __forceinline__ void piece_load(const uint32_t* __restrict__ hrow, uint32_t I, uint32_t i_lo,
                                           const ScoreSmem& s, const psk::RowConst& rc, Piece<NV>& p) {
  const int lane = threadIdx.x & 31;
#pragma unroll
  for (int v = 0; v < NV; ++v) {
    const uint32_t i = i_lo + 128u * v + 4u * lane;
    if (VEC) {
      uint4 x = make_uint4(0u, 0u, 0u, 0u);
      if (i < I) x = __ldg(reinterpret_cast<const uint4*>(hrow + i));
      p.h[v][0] = x.x;
      p.h[v][1] = x.y;
      p.h[v][2] = x.z;
      p.h[v][3] = x.w;
    } else {
#pragma unroll
      for (int k = 0; k < 4; ++k) p.h[v][k] = (i + k < I) ? __ldg(hrow + i + k) : 0u;
    }
  }
  p.amask = 0u;
#pragma unroll
  for (int v = 0; v < NV; ++v) {
    const uint32_t i = i_lo + 128u * v + 4u * lane;
    int32_t rm[4] = {-1, -1, -1, -1};
    if (i < I) lds4(s.room + i, rm);  // padding past I holds -1
#pragma unroll
    for (int k = 0; k < 4; ++k)
      if ((int32_t)rc.L <= rm[k]) p.amask |= 1u << (4 * v + k);
  }
}

template <int NV, bool VEC, bool STASH>
__device__ __forceinline__ uint32_t piece_pass1(const uint32_t* __restrict__ hrow, uint32_t I, uint32_t i_lo,
                                                const ScoreSmem& s, const psk::DevModel& m, const psk::RowConst& rc,
                                                Piece<NV>& p, float* stash, bool all_pairs) {
  const int lane = threadIdx.x & 31;
  piece_load<NV, VEC>(hrow, I, i_lo, s, rc, p);
  uint32_t wbest = 0xFFFFFFFFu;
#pragma unroll
  for (int v = 0; v < NV; ++v) {
    const uint32_t i = i_lo + 128u * v + 4u * lane;
    float tp[4] = {0.0f, 0.0f, 0.0f, 0.0f};
#pragma unroll
    for (int k = 0; k < 4; ++k) {
      const bool inA = (p.amask >> (4 * v + k)) & 1u;
      if (inA || (STASH && all_pairs)) tp[k] = t_pf32(m, rc.L, p.h[v][k]);
      if (inA) wbest = min(wbest, psk::f2ord(__fsub_rn(tp[k], rc.t_cached)));
    }
    if (STASH && i < I) *reinterpret_cast<float4*>(stash + i) = make_float4(tp[0], tp[1], tp[2], tp[3]);
  }
  return wbest;
}

// Pass 2 of a piece: classes, optional per-pair outputs, and the lane's best (key, instance, hit).
// T_pf is evaluated again (the same rounded operations) rather than held in registers.
template <int NV, bool VEC, bool NARROW, bool GEN, bool STASH>
__device__ __forceinline__ void piece_pass2(uint32_t I, uint32_t i_lo, uint64_t x0, const ScoreSmem& s,
                                            const psk::DevModel& m, const psk::RowConst& rc, float wmin,
                                            const Piece<NV>& p, const float* stash, float* __restrict__ tpot_out,
                                            float* __restrict__ ttft_out, uint8_t* __restrict__ cls_out,
                                            uint64_t& bkey, uint32_t& btie, uint32_t& bh) {
  const int lane = threadIdx.x & 31;
  const bool all_pairs = tpot_out || ttft_out || cls_out;
#pragma unroll
  for (int v = 0; v < NV; ++v) {
    const uint32_t i = i_lo + 128u * v + 4u * lane;
    if (i >= I) continue;
    const uint32_t am = (p.amask >> (4 * v)) & 0xFu;
    bool inC[4];
    float tpf[4];
    bool anyC = false;
    if (STASH) {
      const float4 x = *reinterpret_cast<const float4*>(stash + i);
      tpf[0] = x.x;
      tpf[1] = x.y;
      tpf[2] = x.z;
      tpf[3] = x.w;
    }
#pragma unroll
    for (int k = 0; k < 4; ++k) {
      if (!STASH) tpf[k] = (all_pairs || ((am >> k) & 1u)) ? t_pf32(m, rc.L, p.h[v][k]) : 0.0f;
      inC[k] = ((am >> k) & 1u) && psk::pair_in_c(rc, __fsub_rn(tpf[k], rc.t_cached), wmin);
      anyC |= inC[k];
    }
    if (!anyC && !all_pairs) continue;
    float dec0[4], fe[4], tq[4];
    int32_t Bp[4];
    uint64_t k0[4];
    lds4(s.dec0 + i, dec0);
    lds4(s.f + i, fe);
    lds4(s.tq + i, tq);
    lds4(s.Bp + i, Bp);
    lds4(s.k0 + i, k0);
    int32_t q32[4], S32[4];
    int64_t q[4], S[4];
    if (NARROW) {
      lds4(s.q32 + i, q32);
      lds4(s.S32 + i, S32);
    } else {
      lds4(s.q + i, q);
      lds4(s.S + i, S);
    }
    float tp[4], tt[4];
    uint32_t cw = 0u;
#pragma unroll
    for (int k = 0; k < 4; ++k) {
      const int32_t n = (int32_t)rc.L - (int32_t)(p.h[v][k] << 4);
      uint32_t cls = 3u;
      if (all_pairs || inC[k]) {
        if (NARROW) {
          pair_lat32(m, rc, tpf[k], n, dec0[k], fe[k], tq[k], Bp[k], q32[k], S32[k], &tp[k], &tt[k]);
        } else {
          psk::InstTerms it;
          it.dec0 = dec0[k];
          it.f = fe[k];
          it.tq = tq[k];
          it.Bp = Bp[k];
          it.okB = 1;
          psk::PairW x;
          x.tpf = tpf[k];
          x.W = __fsub_rn(x.tpf, rc.t_cached);
          x.n = n;
          x.inA = true;
          psk::pair_lat(m, rc, x, it, q[k], S[k], &tp[k], &tt[k]);
        }
        if ((am >> k) & 1u) cls = inC[k] ? (psk::pair_admitted(m, rc, tp[k], tt[k]) ? 0u : 1u) : 2u;
      }
      cw |= cls << (8 * k);
      if (cls <= 1u) {
        const uint64_t qn = NARROW ? (uint64_t)(uint32_t)(q32[k] + n) : (uint64_t)q[k] + (uint64_t)(int64_t)n;
        const uint32_t h = p.h[v][k];
        uint64_t key;
        uint32_t tie = i + k;
        if (!GEN) {  // Algorithm 1's order: D-C-Q in T, the LMetric product in C \ T
          key = cls == 0u ? psk::packed_key(0u, k0[k] | ((uint64_t)((1u << 26) - 1u - h) << 18))
                          : psk::packed_key(1u, qn * (uint64_t)(uint32_t)Bp[k]);
        } else if (cls == 0u) {
          key = psk::packed_key(0u, psk::value_in_t(m, psk::key0_from_dcq(m, k0[k]), h, tp[k], rc.tpot_target));
          if (m.sel == psk::kSelHCQ) tie |= (uint32_t)(k0[k] & 0x3FFFFull) << 12;
        } else {
          key = psk::packed_key(1u, psk::value_fallback(m, qn, (uint32_t)Bp[k], k0[k], h));
        }
        // a lane's instances ascend, so under the default order ties keep the lowest by themselves
        if (key < bkey || (GEN && key == bkey && tie < btie)) {
          bkey = key;
          btie = tie;
          bh = h;
        }
      }
    }
    if (!all_pairs) continue;
    const uint64_t x = x0 + i;
    if (VEC) {
      if (tpot_out) __stcs(reinterpret_cast<float4*>(tpot_out + x), make_float4(tp[0], tp[1], tp[2], tp[3]));
      if (ttft_out) __stcs(reinterpret_cast<float4*>(ttft_out + x), make_float4(tt[0], tt[1], tt[2], tt[3]));
      if (cls_out) __stcs(reinterpret_cast<uint32_t*>(cls_out + x), cw);
    } else {
#pragma unroll
      for (int k = 0; k < 4; ++k) {
        if (i + k >= I) break;
        if (tpot_out) tpot_out[x + k] = tp[k];
        if (ttft_out) ttft_out[x + k] = tt[k];
        if (cls_out) cls_out[x + k] = (uint8_t)(cw >> (8 * k));
      }
    }
  }
}

constexpr uint32_t kStashMax = 1024;  // rows of up to this many instances keep T_pf in shared memory

template <int NV, bool VEC, bool GEN, bool STASH>
__global__ void __launch_bounds__(kScoreThreads, 2)
score_rows_kernel(const uint32_t* __restrict__ hits, psk::StateSoA st, uint32_t I, psk::WindowDev w,
                  psk::DevModel m, float* __restrict__ tpot_out, float* __restrict__ ttft_out,
                  uint8_t* __restrict__ cls_out, int32_t* __restrict__ best_out,
                  uint8_t* __restrict__ path_out, psk::ShardIO sh) {
  extern __shared__ __align__(16) unsigned long long smem_raw[];
  const uint32_t Ip = (I + 3u) & ~3u;
  const ScoreSmem s = score_smem(smem_raw, Ip);
  // this warp's T_pf row (after the instance arrays), when rows are short enough
  float* const stash = STASH ? reinterpret_cast<float*>(s.S32 + Ip) + (threadIdx.x >> 5) * Ip : nullptr;
  const bool all_pairs = tpot_out || ttft_out || cls_out;
  bool wide = false;  // some instance's q or S is outside [0, 2^30)
  for (uint32_t i = threadIdx.x; i < Ip; i += blockDim.x) {
    if (i < I) {
      const int32_t b = __ldg(st.b + i), qr = __ldg(st.qr + i), Bmax = __ldg(st.Bmax + i);
      const int64_t q = __ldg(st.q + i), S = __ldg(st.S + i), M = __ldg(st.M + i);
      const psk::InstTerms it = psk::inst_terms(m, b, qr, q, Bmax);
      s.q[i] = q;
      s.S[i] = S;
      s.k0[i] = psk::dcq_key0(b, qr);
      s.room[i] = it.okB ? psk::kv_room(S, M) : -1;
      s.dec0[i] = it.dec0;
      s.f[i] = it.f;
      s.tq[i] = it.tq;
      s.Bp[i] = it.Bp;
      wide |= !(q >= 0 && q < (1ll << 30) && S >= 0 && S < (1ll << 30));
      s.q32[i] = (int32_t)q;
      s.S32[i] = (int32_t)S;
    } else {
      s.q[i] = 0;
      s.S[i] = 0;
      s.k0[i] = 0;
      s.room[i] = -1;
      s.dec0[i] = 0.0f;
      s.f[i] = 0.0f;
      s.tq[i] = 0.0f;
      s.Bp[i] = 1;
      s.q32[i] = 0;
      s.S32[i] = 0;
    }
  }
  const bool narrow = __syncthreads_or(wide ? 1 : 0) == 0;
  const int lane = threadIdx.x & 31;
  const uint32_t warps_total = (gridDim.x * blockDim.x) >> 5;
  constexpr uint32_t kPiece = 128u * NV;
  const bool one_piece = I <= kPiece;
  for (uint32_t r = (blockIdx.x * blockDim.x + threadIdx.x) >> 5; r < w.R; r += warps_total) {
    const psk::RowConst rc = psk::row_const(m, __ldg(w.L + r), __ldg(w.ttft_t + r), __ldg(w.tpot_t + r));
    const uint64_t x0 = (uint64_t)r * I;
    const uint32_t* hrow = hits + x0;
    Piece<NV> p;
    uint32_t wbest = piece_pass1<NV, VEC, STASH>(hrow, I, 0u, s, m, rc, p, stash, all_pairs);
    for (uint32_t lo = kPiece; lo < I; lo += kPiece) {
      Piece<NV> p2;
      wbest = min(wbest, piece_pass1<NV, VEC, STASH>(hrow, I, lo, s, m, rc, p2, stash, all_pairs));
    }
    __syncwarp();  // the stash row is read back by other lanes of the warp
    wbest = __reduce_min_sync(0xffffffffu, wbest);
    if (sh.wmin_out) {  // column block, first reduction only
      if (lane == 0) sh.wmin_out[r] = wbest;
      __syncwarp();
      continue;
    }
    if (sh.wmin_in) wbest = __ldg(sh.wmin_in + r);  // the pool's W_min
    const bool anyA = wbest != 0xFFFFFFFFu;  // a W of a pair in A is never NaN, so never all ones
    const float wmin = psk::ord2f(wbest);
    uint64_t bkey = psk::kNoKey;
    uint32_t btie = 0xFFFFFFFFu, bh = 0u;
    if (one_piece) {
      if (narrow)
        piece_pass2<NV, VEC, true, GEN, STASH>(I, 0u, x0, s, m, rc, wmin, p, stash, tpot_out, ttft_out, cls_out, bkey, btie, bh);
      else
        piece_pass2<NV, VEC, false, GEN, STASH>(I, 0u, x0, s, m, rc, wmin, p, stash, tpot_out, ttft_out, cls_out, bkey, btie, bh);
    } else {
      for (uint32_t lo = 0; lo < I; lo += kPiece) {
        if (STASH) piece_load<NV, VEC>(hrow, I, lo, s, rc, p);
        else piece_pass1<NV, VEC, false>(hrow, I, lo, s, m, rc, p, nullptr, all_pairs);
        if (narrow)
          piece_pass2<NV, VEC, true, GEN, STASH>(I, lo, x0, s, m, rc, wmin, p, stash, tpot_out, ttft_out, cls_out, bkey, btie, bh);
        else
          piece_pass2<NV, VEC, false, GEN, STASH>(I, lo, x0, s, m, rc, wmin, p, stash, tpot_out, ttft_out, cls_out, bkey, btie, bh);
      }
    }
    __syncwarp();  // the next row rewrites the stash
    uint64_t key;
    uint32_t tie, hj;
    psk::warp_pick_min(bkey, btie, bh, &key, &tie, &hj);
    if (lane == 0) {
      const bool pick = anyA && key != psk::kNoKey;
      if (best_out) best_out[r] = pick ? (int32_t)(tie & psk::kTieInstMask) : -1;
      if (path_out) path_out[r] = pick ? (uint8_t)(key >> 62) : (uint8_t)2;
      if (sh.key_out) {
        sh.key_out[r] = pick ? key : psk::kNoKey;
        sh.tie_out[r] = pick ? tie + sh.id_base : 0xFFFFFFFFu;
      }
    }
  }
}

// ---- rows of 257 .. 1024 instances: a thread block per row, instance terms in registers ------------
//
// Thread t owns the instances 4t .. 4t + 3 and keeps their request-independent terms in registers
// for the whole launch, so a pair needs no shared-memory load.  A block takes a contiguous range of
// rows, two at a time; their row constants (T_pf(0, L), Z, eta Z, the TTFT budget) are computed once
// per 256 rows into shared memory.  Per pair of rows: each thread loads its four hits of each (16-byte
// loads, the next pair's issued before this pair's work), evaluates pass 1 on both, and the block
// reduces both rows' W_min over A (warp reductions, one barrier, every thread combines the warps'
// values); pass 2 writes the per-pair outputs with 16-byte (TPOT, TTFT) and 4-byte (classes) stores
// and the warps' picks go to shared slots, which one thread per row combines after the next pair's
// barrier.  Shared reduction slots alternate between iterations, so one barrier per pair of rows
// suffices.
constexpr uint32_t kBlkRowsAhead = 256;  // row constants computed per refill
constexpr uint32_t kBlkThreads = 256;    // 4 instances a thread, up to 1024 instances

struct BlkRow {
  float t_cached, Z, etaZ, ttft_budget, tpot_target;
  uint32_t L;
};

template <bool GEN, bool VEC, bool ALL>
__global__ void __launch_bounds__(kBlkThreads, 2)
score_block_kernel(const uint32_t* __restrict__ hits, psk::StateSoA st, uint32_t I, psk::WindowDev w, psk::DevModel m,
                   float* __restrict__ tpot_out, float* __restrict__ ttft_out, uint8_t* __restrict__ cls_out,
                   int32_t* __restrict__ best_out, uint8_t* __restrict__ path_out, psk::ShardIO sh) {
  __shared__ BlkRow s_rc[kBlkRowsAhead];
  __shared__ __align__(16) uint32_t s_w[2][2][8];  // [parity][row of the pair][warp]
  __shared__ unsigned long long s_k[2][2][8];
  __shared__ uint32_t s_t[2][2][8];
  const uint32_t t = threadIdx.x;
  const int lane = (int)(t & 31u), warp = (int)(t >> 5);
  constexpr int nw = kBlkThreads / 32;  // the launch's block size
  const uint32_t i0 = 4u * t;
  constexpr bool all_pairs = ALL;  // some per-pair output is wanted (the launch checks)
  // instance terms (padding instances past I fail the capacity guard: room -1)
  int32_t room[4], q32[4], S32[4], Bp[4];
  float dec0[4], fe[4], tq[4];
  uint64_t k0[4];
  bool wide = false;
#pragma unroll
  for (int k = 0; k < 4; ++k) {
    const uint32_t i = i0 + (uint32_t)k;
    room[k] = -1;
    q32[k] = S32[k] = 0;
    Bp[k] = 1;
    dec0[k] = fe[k] = tq[k] = 0.0f;
    k0[k] = 0ull;
    if (i < I) {
      const int32_t b = __ldg(st.b + i), qr = __ldg(st.qr + i), Bmax = __ldg(st.Bmax + i);
      const int64_t q = __ldg(st.q + i), S = __ldg(st.S + i), M = __ldg(st.M + i);
      const psk::InstTerms it = psk::inst_terms(m, b, qr, q, Bmax);
      room[k] = it.okB ? psk::kv_room(S, M) : -1;
      dec0[k] = it.dec0;
      fe[k] = it.f;
      tq[k] = it.tq;
      Bp[k] = it.Bp;
      k0[k] = psk::dcq_key0(b, qr);
      wide |= !(q >= 0 && q < (1ll << 30) && S >= 0 && S < (1ll << 30));
      q32[k] = (int32_t)q;
      S32[k] = (int32_t)S;
    }
  }
  // every instance's q and S below 2^30: the 32-bit sums are exact (else 64-bit state per pair)
  const bool narrow = __syncthreads_or(wide ? 1 : 0) == 0;
  // the row loop, compiled for the narrow and the wide state separately (a block-uniform choice)
  auto rows_loop = [&](auto narrow_tag) {
    constexpr bool NARROW = decltype(narrow_tag)::value;
    const uint32_t per = (w.R + gridDim.x - 1) / gridDim.x;
    const uint32_t r_lo = blockIdx.x * per;
    const uint32_t r_hi = min(w.R, r_lo + per);
    auto load_hits = [&](uint32_t r, uint32_t (&h)[4]) {
      const uint32_t* hrow = hits + (uint64_t)r * I;
      if (VEC) {
        uint4 x = make_uint4(0u, 0u, 0u, 0u);
        if (i0 < I) x = __ldcs(reinterpret_cast<const uint4*>(hrow + i0));
        h[0] = x.x;
        h[1] = x.y;
        h[2] = x.z;
        h[3] = x.w;
      } else {
#pragma unroll
        for (int k = 0; k < 4; ++k) h[k] = (i0 + k < I) ? __ldcs(hrow + i0 + k) : 0u;
      }
    };
    auto rc_of = [&](uint32_t rr) {
      const BlkRow& b = s_rc[rr];
      psk::RowConst rc;
      rc.t_cached = b.t_cached;
      rc.Z = b.Z;
      rc.etaZ = b.etaZ;
      rc.ttft_budget = b.ttft_budget;
      rc.tpot_target = b.tpot_target;
      rc.L = b.L;
      return rc;
    };
    // pass 1 of a row: capacity guard, T_pf at the hit, this thread's W_min over A.  T_pf depends on
    // the row and the hit only, and most of a row's instances share a hit (the shared system prompt),
    // so a thread evaluates it at its first instance's hit and again only where a hit differs (a
    // warp-uniform test: the warp skips the evaluation when no lane's hit differs).
    auto pass1 = [&](const psk::RowConst& rc, const uint32_t (&h)[4], float (&tp)[4], uint32_t& am) {
      uint32_t wbest = 0xFFFFFFFFu;
      am = 0u;
      const float tb = t_pf32(m, rc.L, h[0]);
#pragma unroll
      for (int k = 0; k < 4; ++k) {
        const bool inA = (int32_t)rc.L <= room[k];
        am |= (inA ? 1u : 0u) << k;
        tp[k] = tb;
        const bool other = h[k] != h[0] && (inA || all_pairs);
        if (k > 0 && __any_sync(0xffffffffu, other)) {
          if (other) tp[k] = t_pf32(m, rc.L, h[k]);
        }
        if (inA) wbest = min(wbest, psk::f2ord(__fsub_rn(tp[k], rc.t_cached)));
      }
      return wbest;
    };
    // pass 2 of row r: classes, latencies, the per-pair outputs, this thread's best (key, tie)
    auto pass2 = [&](uint32_t r, const psk::RowConst& rc, const uint32_t (&h)[4], const float (&tp)[4], uint32_t am,
                     float wmin, uint64_t& bkey, uint32_t& btie) {
      bkey = psk::kNoKey;
      btie = 0xFFFFFFFFu;
      float to[4], tt[4];
      uint32_t cw = 0u;
#pragma unroll
      for (int k = 0; k < 4; ++k) {
        const uint32_t i = i0 + (uint32_t)k;
        const bool inA = (am >> k) & 1u;
        const bool inC = inA && psk::pair_in_c(rc, __fsub_rn(tp[k], rc.t_cached), wmin);
        const int32_t n = (int32_t)rc.L - (int32_t)(h[k] << 4);
        to[k] = tt[k] = 0.0f;
        uint32_t cls = 3u;
        if (all_pairs || inC) {
          if (NARROW) {
            pair_lat32(m, rc, tp[k], n, dec0[k], fe[k], tq[k], Bp[k], q32[k], S32[k], &to[k], &tt[k]);
          } else if (i < I) {
            psk::InstTerms it;
            it.dec0 = dec0[k];
            it.f = fe[k];
            it.tq = tq[k];
            it.Bp = Bp[k];
            it.okB = 1;
            psk::PairW x;
            x.tpf = tp[k];
            x.W = __fsub_rn(x.tpf, rc.t_cached);
            x.n = n;
            x.inA = true;
            psk::pair_lat(m, rc, x, it, __ldg(st.q + i), __ldg(st.S + i), &to[k], &tt[k]);
          }
          if (inA) cls = inC ? (psk::pair_admitted(m, rc, to[k], tt[k]) ? 0u : 1u) : 2u;
        }
        cw |= cls << (8 * k);
        if (cls <= 1u) {
          const uint64_t qn = NARROW ? (uint64_t)(uint32_t)(q32[k] + n)
                                     : (uint64_t)__ldg(st.q + i) + (uint64_t)(int64_t)n;
          uint64_t key;
          uint32_t tie = i;
          if (!GEN) {
            key = cls == 0u ? psk::packed_key(0u, k0[k] | ((uint64_t)((1u << 26) - 1u - h[k]) << 18))
                            : psk::packed_key(1u, qn * (uint64_t)(uint32_t)Bp[k]);
          } else if (cls == 0u) {
            key = psk::packed_key(0u, psk::value_in_t(m, psk::key0_from_dcq(m, k0[k]), h[k], to[k], rc.tpot_target));
            if (m.sel == psk::kSelHCQ) tie |= (uint32_t)(k0[k] & 0x3FFFFull) << 12;
          } else {
            key = psk::packed_key(1u, psk::value_fallback(m, qn, (uint32_t)Bp[k], k0[k], h[k]));
          }
          if (key < bkey || (GEN && key == bkey && tie < btie)) {  // this thread's instances ascend
            bkey = key;
            btie = tie;
          }
        }
      }
      if (all_pairs && i0 < I) {
        const uint64_t x = (uint64_t)r * I + i0;
        if (VEC) {
          if (tpot_out) __stcs(reinterpret_cast<float4*>(tpot_out + x), make_float4(to[0], to[1], to[2], to[3]));
          if (ttft_out) __stcs(reinterpret_cast<float4*>(ttft_out + x), make_float4(tt[0], tt[1], tt[2], tt[3]));
          if (cls_out) __stcs(reinterpret_cast<uint32_t*>(cls_out + x), cw);
        } else {
#pragma unroll
          for (int k = 0; k < 4; ++k) {
            if (i0 + k >= I) break;
            if (tpot_out) tpot_out[x + k] = to[k];
            if (ttft_out) ttft_out[x + k] = tt[k];
            if (cls_out) cls_out[x + k] = (uint8_t)(cw >> (8 * k));
          }
        }
      }
    };
    // Rows two at a time: both rows' W_min in one barrier.  The picks of a pair of rows are combined
    // after the next pair's barrier (their slots alternate between iterations), so an iteration has
    // one barrier.
    auto merge = [&](uint32_t rp, int q, uint32_t pw, uint32_t pp) {
      // row rp's pick from the warps' (key, tie) in slot s_k[pp][q]
      uint64_t kb = psk::kNoKey;
      uint32_t tb = 0xFFFFFFFFu;
      for (int v = 0; v < nw; ++v) {
        const uint64_t kv = s_k[pp][q][v];
        const uint32_t tv = s_t[pp][q][v];
        if (kv < kb || (kv == kb && tv < tb)) {
          kb = kv;
          tb = tv;
        }
      }
      const bool pick = pw != 0xFFFFFFFFu && kb != psk::kNoKey;
      if (best_out) best_out[rp] = pick ? (int32_t)(tb & psk::kTieInstMask) : -1;
      if (path_out) path_out[rp] = pick ? (uint8_t)(kb >> 62) : (uint8_t)2;
      if (sh.key_out) {
        sh.key_out[rp] = pick ? kb : psk::kNoKey;
        sh.tie_out[rp] = pick ? tb + sh.id_base : 0xFFFFFFFFu;
      }
    };
    uint32_t hn[2][4] = {{0u, 0u, 0u, 0u}, {0u, 0u, 0u, 0u}};
    if (r_lo < r_hi) load_hits(r_lo, hn[0]);
    if (r_lo + 1 < r_hi) load_hits(r_lo + 1, hn[1]);
    uint32_t par = 0;
    bool prev = false;          // a pair of rows whose picks are still to be combined
    uint32_t prev_r = 0, pw0 = 0u, pw1 = 0u;
    bool prev_two = false;
    for (uint32_t r = r_lo; r < r_hi; r += 2, par ^= 1u) {
      const bool two = r + 1 < r_hi;
      const uint32_t rr = (r - r_lo) % kBlkRowsAhead;  // even, so row r + 1 is in the same batch
      if (rr == 0) {
        __syncthreads();  // every thread is done with the previous batch of row constants
        const uint32_t x = r + t;
        if (t < kBlkRowsAhead && x < r_hi) {
          const psk::RowConst rc = psk::row_const(m, __ldg(w.L + x), __ldg(w.ttft_t + x), __ldg(w.tpot_t + x));
          s_rc[t] = BlkRow{rc.t_cached, rc.Z, rc.etaZ, rc.ttft_budget, rc.tpot_target, rc.L};
        }
        __syncthreads();
      }
      const psk::RowConst rc0 = rc_of(rr);
      const psk::RowConst rc1 = rc_of(two ? rr + 1 : rr);
      uint32_t h0[4], h1[4];
#pragma unroll
      for (int k = 0; k < 4; ++k) {
        h0[k] = hn[0][k];
        h1[k] = hn[1][k];
      }
      if (r + 2 < r_hi) load_hits(r + 2, hn[0]);  // in flight during these rows
      if (r + 3 < r_hi) load_hits(r + 3, hn[1]);
      float tp0[4], tp1[4];
      uint32_t am0, am1;
      uint32_t w0 = pass1(rc0, h0, tp0, am0);
      uint32_t w1 = two ? pass1(rc1, h1, tp1, am1) : 0xFFFFFFFFu;
      if (!two) {
        am1 = 0u;
#pragma unroll
        for (int k = 0; k < 4; ++k) tp1[k] = 0.0f;
      }
      w0 = __reduce_min_sync(0xffffffffu, w0);
      w1 = __reduce_min_sync(0xffffffffu, w1);
      if (lane == 0) {
        s_w[par][0][warp] = w0;
        s_w[par][1][warp] = w1;
      }
      __syncthreads();
      // the previous pair's picks (its warps' slots were written before this barrier)
      if (prev && (t == 0 || (t == 32 && prev_two))) {
        const int q = t == 0 ? 0 : 1;
        merge(prev_r + (uint32_t)q, q, q == 0 ? pw0 : pw1, par ^ 1u);
      }
      {  // the eight warps' values of both rows, four 16-byte loads
        const uint4* sw = reinterpret_cast<const uint4*>(&s_w[par][0][0]);
        const uint4 a0 = sw[0], a1 = sw[1], b0 = sw[2], b1 = sw[3];
        w0 = min(min(min(a0.x, a0.y), min(a0.z, a0.w)), min(min(a1.x, a1.y), min(a1.z, a1.w)));
        w1 = min(min(min(b0.x, b0.y), min(b0.z, b0.w)), min(min(b1.x, b1.y), min(b1.z, b1.w)));
      }
      if (sh.wmin_out) {  // column block, first reduction only
        if (t == 0) sh.wmin_out[r] = w0;
        if (t == 32 && two) sh.wmin_out[r + 1] = w1;
        continue;
      }
      if (sh.wmin_in) {  // the pool's W_min
        w0 = __ldg(sh.wmin_in + r);
        if (two) w1 = __ldg(sh.wmin_in + r + 1);
      }
      uint64_t bk0, bk1 = psk::kNoKey;
      uint32_t bt0, bt1 = 0xFFFFFFFFu;
      pass2(r, rc0, h0, tp0, am0, psk::ord2f(w0), bk0, bt0);
      if (two) pass2(r + 1, rc1, h1, tp1, am1, psk::ord2f(w1), bk1, bt1);
      uint64_t key0, key1;
      uint32_t tie0, tie1, hj;
      psk::warp_pick_min(bk0, bt0, 0u, &key0, &tie0, &hj);
      psk::warp_pick_min(bk1, bt1, 0u, &key1, &tie1, &hj);
      if (lane == 0) {
        s_k[par][0][warp] = key0;
        s_t[par][0][warp] = tie0;
        s_k[par][1][warp] = key1;
        s_t[par][1][warp] = tie1;
      }
      prev = true;
      prev_r = r;
      prev_two = two;
      pw0 = w0;
      pw1 = w1;
    }
    __syncthreads();
    if (prev && (t == 0 || (t == 32 && prev_two))) {
      const int q = t == 0 ? 0 : 1;
      merge(prev_r + (uint32_t)q, q, q == 0 ? pw0 : pw1, par ^ 1u);
    }
  };
  if (narrow) rows_loop(std::integral_constant<bool, true>());
  else rows_loop(std::integral_constant<bool, false>());
}

cudaError_t score_block_launch(const uint32_t* hits, psk::StateSoA st, uint32_t I, const psk::WindowDev& w,
                               const psk::DevModel& m, float* tpot, float* ttft, uint8_t* cls, int32_t* best,
                               uint8_t* path, int num_sms, cudaStream_t s, const psk::ShardIO& sh) {
  const bool vec = (I & 3u) == 0u && (reinterpret_cast<uintptr_t>(hits) & 15u) == 0u &&
                   (reinterpret_cast<uintptr_t>(tpot) & 15u) == 0u && (reinterpret_cast<uintptr_t>(ttft) & 15u) == 0u &&
                   (reinterpret_cast<uintptr_t>(cls) & 3u) == 0u;
  const bool gen = m.sel != psk::kSelDCQ || m.fb_dcq;
  const uint32_t threads = kBlkThreads;
  const bool all = tpot || ttft || cls;
  decltype(&score_block_kernel<true, true, true>) kern;
  if (all)
    kern = vec ? (gen ? score_block_kernel<true, true, true> : score_block_kernel<false, true, true>)
               : (gen ? score_block_kernel<true, false, true> : score_block_kernel<false, false, true>);
  else
    kern = vec ? (gen ? score_block_kernel<true, true, false> : score_block_kernel<false, true, false>)
               : (gen ? score_block_kernel<true, false, false> : score_block_kernel<false, false, false>);
  int per_sm = 0;  // one wave of resident blocks, each taking a contiguous range of rows
  cudaError_t e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, kern, (int)threads, 0);
  if (e != cudaSuccess) return e;
  uint32_t grid = (uint32_t)num_sms * (uint32_t)(per_sm > 0 ? per_sm : 1);
  if (grid > w.R) grid = w.R;
  kern<<<grid, threads, 0, s>>>(hits, st, I, w, m, tpot, ttft, cls, best, path, sh);
  return cudaGetLastError();
}

template <int NV>
cudaError_t score_launch(const uint32_t* hits, psk::StateSoA st, uint32_t I, const psk::WindowDev& w,
                         const psk::DevModel& m, float* tpot, float* ttft, uint8_t* cls, int32_t* best,
                         uint8_t* path, int num_sms, cudaStream_t s, const psk::ShardIO& sh) {
  const uint32_t Ip = (I + 3u) & ~3u;
  size_t smem = (size_t)Ip * (3 * sizeof(int64_t) + 7 * sizeof(uint32_t));
  if (Ip <= kStashMax) smem += (size_t)(kScoreThreads / 32) * Ip * sizeof(float);
  // 16-byte loads of hit rows and stores of TPOT / TTFT rows, 4-byte stores of class rows
  const bool vec = (I & 3u) == 0u && (reinterpret_cast<uintptr_t>(hits) & 15u) == 0u &&
                   (reinterpret_cast<uintptr_t>(tpot) & 15u) == 0u && (reinterpret_cast<uintptr_t>(ttft) & 15u) == 0u &&
                   (reinterpret_cast<uintptr_t>(cls) & 3u) == 0u;
  const bool gen = m.sel != psk::kSelDCQ || m.fb_dcq;  // not Algorithm 1's order (Table 4 / Table 3 variants)
  // rows of up to kStashMax instances (every NV < 4 window) keep T_pf in shared memory
  constexpr bool kCanSkipStash = NV == 4;
  const bool stash = Ip <= kStashMax || !kCanSkipStash;
  decltype(&score_rows_kernel<NV, true, true, true>) kern;
  if (stash)
    kern = vec ? (gen ? score_rows_kernel<NV, true, true, true> : score_rows_kernel<NV, true, false, true>)
               : (gen ? score_rows_kernel<NV, false, true, true> : score_rows_kernel<NV, false, false, true>);
  else
    kern = vec ? (gen ? score_rows_kernel<NV, true, true, kCanSkipStash ? false : true>
                      : score_rows_kernel<NV, true, false, kCanSkipStash ? false : true>)
               : (gen ? score_rows_kernel<NV, false, true, kCanSkipStash ? false : true>
                      : score_rows_kernel<NV, false, false, kCanSkipStash ? false : true>);
  cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (e != cudaSuccess) return e;
  const uint32_t rows_per_block = kScoreThreads / 32;
  uint32_t grid = (w.R + rows_per_block - 1) / rows_per_block;
  const uint32_t cap = (uint32_t)num_sms * 2u;
  if (grid > cap) grid = cap;
  kern<<<grid, kScoreThreads, smem, s>>>(hits, st, I, w, m, tpot, ttft, cls, best, path, sh);
  return cudaGetLastError();
}

}  // namespace

namespace pskl {

cudaError_t launch_score(const uint32_t* hits, psk::StateSoA st, uint32_t I, const psk::WindowDev& w,
                         const psk::DevModel& m, float* tpot, float* ttft, uint8_t* cls, int32_t* best,
                         uint8_t* path, int num_sms, cudaStream_t s, const psk::ShardIO& sh) {
  if (w.R == 0) return cudaSuccess;
  if (I <= 128u) return score_launch<1>(hits, st, I, w, m, tpot, ttft, cls, best, path, num_sms, s, sh);
  if (I <= 256u) return score_launch<2>(hits, st, I, w, m, tpot, ttft, cls, best, path, num_sms, s, sh);
  if (I <= 1024u) return score_block_launch(hits, st, I, w, m, tpot, ttft, cls, best, path, num_sms, s, sh);
  return score_launch<4>(hits, st, I, w, m, tpot, ttft, cls, best, path, num_sms, s, sh);
}

}  // namespace pskl
