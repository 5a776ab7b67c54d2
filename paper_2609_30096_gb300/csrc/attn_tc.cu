// Flash attention on the sm_103a tensor cores (bf16 in, fp32 accumulate):
// O = softmax(Q K^T / sqrt(hd)) V per (sequence, head), no mask.
//
// Two kernels share the schedules below: k_attn_tc, whose work item is one
// 128-query tile (described first), and k_attn_pp, whose item is a pair of
// query tiles sharing every K/V tile (described before it, further down; the
// default).
//
// Work: an item is one 128-query tile of one (sequence, head); its KT key tiles
// of 128 keys are its units.  The kernel is persistent (at most one CTA per SM)
// and follows one of two schedules:
//   data-parallel  CTA w takes items w, w + G, ... with all their key tiles;
//   stream-K       the items' key tiles form one sequence of U units and CTA w
//                  takes the contiguous share [w U / G, (w+1) U / G), so every
//                  SM processes the same number of key tiles whatever the item
//                  count.  A query tile split across CTAs is finished by
//                  whichever part ends last: the others publish their running
//                  row maximum m, row sum l and unnormalized O (fp32) to a
//                  workspace slot and count in on a per-(item, warp) counter;
//                  the last one combines the parts in key order,
//                  O = sum_p 2^(m_p - M) O_p / sum_p 2^(m_p - M) l_p with
//                  M = max_p m_p (a fixed order: the bits do not depend on
//                  timing), writes the output and resets the counter.
// A CTA walks its segments (item, first key tile, end key tile) with 320
// threads:
//   warp 0      TMA: lane 0 the Q tile of each segment (two buffers) and the K
//               tiles (three-stage ring), lane 1 the V tiles (two-stage ring);
//               4-D tensor maps over head-major or token-major operands,
//               128-byte swizzle, zero fill past L.
//   warp 1      allocates TMEM (two O accumulators of hd columns, two
//               128-column S buffers) and issues, from one thread,
//               S(j+1) = Q K(j+1)^T (possibly the next segment's first tile)
//               while the softmax warps work on S(j), then O += P(j) V(j)
//               into the segment's O buffer.  P is read from TMEM (the A
//               operand), V is the MN-major B operand from shared memory.
//   warps 2-9   softmax, two warpgroups splitting each key tile by columns (64
//               keys each), one thread per query row (its TMEM lane): row
//               maximum over the valid keys (halves combined through shared
//               memory), lazy rescaling of O (only when the running maximum
//               grows by more than 2^8), P = exp2(S log2(e)/sqrt(hd) - m)
//               rounded to bf16 pairs and written over the first 32 of the
//               group's 64 S columns, and at the end of a segment the output
//               (or the stream-K publish / combine).  O is double-buffered, so
//               the next segment's MMAs run while a segment's output is read.
// Tensor-core operations issued by one thread execute in issue order, so
// S(j+2), issued after O += P(j) V(j), overwrites P(j) only after it was read.
// Every mbarrier wait is bounded (see tc_common.cuh).
#include <cuda.h>
#include <cuda_bf16.h>
#include <math.h>

#include <atomic>

#include "internal.h"
#include "tc_common.cuh"

namespace track {

namespace {

using namespace tc;
typedef __nv_bfloat16 bf16;

constexpr int AT_BM = 128;        // query rows per item (MMA M)
constexpr int AT_BN = 128;        // keys per tile
constexpr int AT_KH = AT_BN / 2;  // keys per softmax group
constexpr int AT_THREADS = 320;   // warp 0 TMA, warp 1 MMA, warps 2-9 softmax
constexpr int AT_MAX_PARTS = 4;   // the host only picks stream-K when no item spans more CTAs

template <int HD>
struct AtShape {
  static constexpr uint32_t Q_BYTES = AT_BM * HD * 2;   // HD/64 boxes of [128 rows][128 B]
  static constexpr uint32_t KV_BYTES = AT_BN * HD * 2;  // one K or V tile
  static constexpr uint32_t X_BYTES = 2 * 2 * AT_BM * 4;  // row partials [parity][half][row]
  static constexpr int KST = 3;  // K ring stages (V: 2)
  // The dynamic shared window starts 1024-byte aligned (after the reserved
  // 1 KB); the kernel checks that before its first copy.
  static constexpr size_t SMEM = 2 * Q_BYTES + (KST + 2) * (size_t)KV_BYTES + X_BYTES + 256;
  // TMEM columns: O buffer b at b*HD, S buffer b at TM_S0 + 128 b
  static constexpr uint32_t TM_S0 = 2 * HD;
  static constexpr uint32_t TMEM_COLS = 512;
  static_assert(TM_S0 + 2 * AT_BN <= TMEM_COLS, "TMEM budget");
  // Stream-K slot: per softmax warp, its 32 rows x HD/2 columns of O (float4
  // index (w * HD/8 + j) * 32 + lane), then per warp m[32] and l[32].
  static constexpr int SLOT = AT_BM * HD + 8 * 2 * 32;
};

struct AtSk {
  int* cnt;       // [8 * items] counters, zero between launches (nullptr: data-parallel)
  float* ws;      // [2 * G] slots
  int64_t units;  // items * key tiles
};

// The descriptor of the operand starting `bytes` (a multiple of 16) after the one
// `d` describes: the start-address field holds the shared address / 16 in its
// low 14 bits, and shared-memory addresses stay below 2^18, so adding bytes / 16
// never carries into the next field.
__device__ __forceinline__ uint64_t sdesc_add(uint64_t d, uint32_t bytes) {
  return d + (uint64_t)(bytes >> 4);
}

__device__ __forceinline__ uint32_t pack_bf16x2(float lo, float hi) {
  __nv_bfloat162 t = __floats2bfloat162_rn(lo, hi);
  return *reinterpret_cast<uint32_t*>(&t);
}

// Loads a box of rows l0.. (64 columns from col) of head h of sequence sq; the
// tensor map's dimensions are (hd, H, L, S) for a token-major operand and
// (hd, L, H, S) for a head-major one.
__device__ __forceinline__ void tma_load_rows(uint32_t dst, const CUtensorMap* tm, int tok, int col,
                                              int l0, int h, int sq, uint32_t bar) {
  if (tok) tma_load_4d(dst, tm, col, h, l0, sq, bar);
  else tma_load_4d(dst, tm, col, l0, h, sq, bar);
}

// Lane 0 waits, the whole warp learns the outcome.
__device__ __forceinline__ bool warp_wait(uint32_t bar, uint32_t parity, volatile int* abort_flag,
                                          int* err, int code) {
  int ok = 1;
  if ((threadIdx.x & 31) == 0) ok = mbar_wait(bar, parity, abort_flag, err, code) ? 1 : 0;
  return __shfl_sync(0xffffffffu, ok, 0) != 0;
}

// Output of a segment's query tile, by one softmax warp (its 32 rows, columns
// half*HD/2 ..): O / l for a whole item; for a stream-K part, publish (m, l, O)
// or, as the last part, combine all parts in key order.  (Inlined: a call here
// measured 1.5 % slower per key tile.)  tO addresses this
// warp's lanes and columns of the segment's O buffer.  False if the item
// spans more CTAs than the kernel supports (excluded by the host).
template <int HD>
__device__ __forceinline__ bool segment_output(uint32_t tO, float m, float lt, int item, int kt0,
                                            int kt1, int KT, int QT, int H, int Lq, int64_t U,
                                            bf16* __restrict__ O, int half, int row, int lane,
                                            int wi, const AtSk& sk, int* err,
                                            volatile int* abort_flag) {
  using S = AtShape<HD>;
  // Writes 32 output columns (row-normalized by inv) of this thread's row.
  auto store32 = [&](bf16* dst, const float (&v)[32], float inv) {
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      uint4 u;
      u.x = pack_bf16x2(v[8 * j] * inv, v[8 * j + 1] * inv);
      u.y = pack_bf16x2(v[8 * j + 2] * inv, v[8 * j + 3] * inv);
      u.z = pack_bf16x2(v[8 * j + 4] * inv, v[8 * j + 5] * inv);
      u.w = pack_bf16x2(v[8 * j + 6] * inv, v[8 * j + 7] * inv);
      *reinterpret_cast<uint4*>(dst + 8 * j) = u;
    }
  };
  const int bh = item / QT, sq = bh / H, hq = bh % H;
  const int qrow = (item % QT) * AT_BM + row;
  bf16* orow = O + (((int64_t)sq * Lq + qrow) * H + hq) * HD + half * (HD / 2);
  if (kt0 == 0 && kt1 == KT) {
    // The whole item: O / l.
    const float inv = 1.f / lt;
#pragma unroll 1
    for (int cc = 0; cc < HD / 64; ++cc) {
      uint32_t r[32];
      tmem_ld32(tO + cc * 32, r);
      float v[32];
#pragma unroll
      for (int t = 0; t < 32; ++t) v[t] = __uint_as_float(r[t]);
      if (qrow < Lq) store32(orow + cc * 32, v, inv);
    }
  } else {
    // Stream-K part of an item split across CTAs.
    const int64_t iu = (int64_t)item * KT;
    const int w_first = sk_worker_of(iu, U, gridDim.x);
    const int nparts = sk_worker_of(iu + KT - 1, U, gridDim.x) - w_first + 1;
    const int part = (int)blockIdx.x - w_first;
    if (nparts > AT_MAX_PARTS) {  // excluded by the host's choice of schedule
      if (lane == 0) {
        *abort_flag = 1;
        atomicExch(err, 24);
      }
      return false;
    }
    // Slot of part i: 2w for worker w's first segment, 2w+1 for its last.
    auto slot_of = [&](int i) -> float* {
      const int wk = w_first + i;
      const int first_item = (int)(((int64_t)wk * U / gridDim.x) / KT);
      return sk.ws + (size_t)(2 * wk + (first_item == item ? 0 : 1)) * S::SLOT;
    };
    int* cnt = sk.cnt + 8 * item + wi;
    int last = 0;
    if (lane == 0) last = ld_acquire(cnt) == nparts - 1 ? 1 : 0;
    last = __shfl_sync(0xffffffffu, last, 0);
    if (!last) {
      // Publish m, l and this warp's 32 rows x HD/2 columns of O.
      float* mine = slot_of(part);
      float4* o4 = reinterpret_cast<float4*>(mine) + (size_t)wi * (HD / 8) * 32 + lane;
#pragma unroll 1
      for (int cc = 0; cc < HD / 64; ++cc) {
        uint32_t r[32];
        tmem_ld32(tO + cc * 32, r);
#pragma unroll
        for (int j = 0; j < 8; ++j)
          o4[(cc * 8 + j) * 32] =
              make_float4(__uint_as_float(r[4 * j]), __uint_as_float(r[4 * j + 1]),
                          __uint_as_float(r[4 * j + 2]), __uint_as_float(r[4 * j + 3]));
      }
      float* ml = mine + AT_BM * HD + wi * 64;
      ml[lane] = m;
      ml[32 + lane] = lt;
      __threadfence();
      __syncwarp();
      if (lane == 0) last = atomicAdd(cnt, 1) == nparts - 1 ? 1 : 0;
      last = __shfl_sync(0xffffffffu, last, 0);
    }
    if (last) {
      __threadfence();  // the other parts' stores are visible to this warp's loads
      if (lane == 0) *cnt = 0;  // every part has counted in: reset for the next launch
      // Weights 2^(m_p - M) and the combined row sum, parts in key order.
      float wp[AT_MAX_PARTS], lp[AT_MAX_PARTS];
      float M = m;
#pragma unroll
      for (int i = 0; i < AT_MAX_PARTS; ++i) {
        wp[i] = -INFINITY;
        lp[i] = 0.f;
        if (i < nparts) {
          if (i == part) {
            wp[i] = m;
            lp[i] = lt;
          } else {
            const float* ml = slot_of(i) + AT_BM * HD + wi * 64;
            wp[i] = __ldcg(ml + lane);
            lp[i] = __ldcg(ml + 32 + lane);
          }
          M = fmaxf(M, wp[i]);
        }
      }
      float den = 0.f;
#pragma unroll
      for (int i = 0; i < AT_MAX_PARTS; ++i) {
        wp[i] = i < nparts ? exp2_approx(wp[i] - M) : 0.f;
        den = fmaf(wp[i], lp[i], den);
      }
      const float inv = 1.f / den;
#pragma unroll 1
      for (int cc = 0; cc < HD / 64; ++cc) {
        uint32_t r[32];
        tmem_ld32(tO + cc * 32, r);
        float acc[32];
#pragma unroll
        for (int t = 0; t < 32; ++t) acc[t] = 0.f;
#pragma unroll
        for (int i = 0; i < AT_MAX_PARTS; ++i) {
          if (i >= nparts) break;
          float x[32];
          if (i == part) {
#pragma unroll
            for (int t = 0; t < 32; ++t) x[t] = __uint_as_float(r[t]);
          } else {
            const float4* src = reinterpret_cast<const float4*>(slot_of(i)) +
                                (size_t)wi * (HD / 8) * 32 + lane;
#pragma unroll
            for (int j = 0; j < 8; ++j) {
              const float4 q = __ldcg(src + (cc * 8 + j) * 32);
              x[4 * j] = q.x; x[4 * j + 1] = q.y; x[4 * j + 2] = q.z; x[4 * j + 3] = q.w;
            }
          }
#pragma unroll
          for (int t = 0; t < 32; ++t) acc[t] = fmaf(wp[i], x[t], acc[t]);
        }
        if (qrow < Lq) store32(orow + cc * 32, acc, inv);
      }
    }
  }
  return true;
}

template <int HD>
__global__ void __launch_bounds__(AT_THREADS, 1)
    k_attn_tc(const __grid_constant__ CUtensorMap tmQ, const __grid_constant__ CUtensorMap tmK,
              const __grid_constant__ CUtensorMap tmV, bf16* __restrict__ O, int H, int Lq, int Lk,
              float scale_log2, int q_tok, int kv_tok, int* err, int items, const AtSk sk) {
  using S = AtShape<HD>;
  constexpr int NB = HD / 64;  // 64-column boxes per row of Q/K/V
  extern __shared__ __align__(1024) uint8_t smem_raw[];
  uint8_t* smem = smem_raw;
  uint8_t* sQ = smem;                         // [2] Q buffers
  uint8_t* sK = sQ + 2 * S::Q_BYTES;          // [3] K stages
  uint8_t* sV = sK + S::KST * S::KV_BYTES;    // [2] V stages
  float* xch = (float*)(sV + 2 * S::KV_BYTES);  // [2][2][AT_BM] row partials
  uint64_t* bars = (uint64_t*)((uint8_t*)xch + S::X_BYTES);
  uint64_t* q_full = bars;        // [2] per Q buffer
  uint64_t* q_empty = bars + 2;   // [2] freed once the segment's last S MMA completed
  uint64_t* k_full = bars + 4;    // [3] per K stage
  uint64_t* k_empty = bars + 7;   // [3] freed once S = Q K^T of the tile has completed
  uint64_t* v_full = bars + 10;   // [2] per V stage
  uint64_t* v_empty = bars + 12;  // [2] freed once P V of the tile has completed
  uint64_t* s_full = bars + 14;   // [2] per S buffer
  uint64_t* p_full = bars + 16;   // [2] P of the tile written into its S buffer (8 softmax warps)
  uint64_t* o_done = bars + 18;   // P V of the tile has completed
  uint64_t* o_full = bars + 19;   // [2] every P V of the segment in this O buffer has completed
  uint64_t* o_empty = bars + 21;  // [2] the segment's output was read out of this O buffer (8 warps)
  uint64_t* xbar = bars + 23;     // [2] all 8 softmax warps' row partials written (per parity)
  uint64_t* done = bars + 25;     // every MMA of the CTA has completed
  uint32_t* tmem_slot = (uint32_t*)(bars + 26);
  volatile int* abort_flag = (volatile int*)(tmem_slot + 1);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int QT = (Lq + AT_BM - 1) / AT_BM, KT = (Lk + AT_BN - 1) / AT_BN;
  const bool use_sk = sk.cnt != nullptr;
  const int64_t U = use_sk ? sk.units : (int64_t)items * KT;

  if (threadIdx.x == 0) {
    for (int i = 0; i < S::KST; ++i) {
      mbar_init(su32(&k_full[i]), 1);
      mbar_init(su32(&k_empty[i]), 1);
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(su32(&q_full[i]), 1);
      mbar_init(su32(&q_empty[i]), 1);
      mbar_init(su32(&v_full[i]), 1);
      mbar_init(su32(&v_empty[i]), 1);
      mbar_init(su32(&s_full[i]), 1);
      mbar_init(su32(&p_full[i]), 8);
      mbar_init(su32(&o_full[i]), 1);
      mbar_init(su32(&o_empty[i]), 8);
      mbar_init(su32(&xbar[i]), 8);
    }
    mbar_init(su32(o_done), 1);
    mbar_init(su32(done), 1);
    *abort_flag = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  if (warp == 1) tmem_alloc(su32(tmem_slot), S::TMEM_COLS);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem_base = *tmem_slot;
  // The prologue above overlaps the previous kernel; inputs and outputs are touched only now.
  pdl_wait();
  pdl_release();
  if ((su32(smem) & 1023u) != 0) {  // the 128-byte-swizzled tiles need 1024-byte alignment
    if (threadIdx.x == 0) atomicExch(err, 25);
    __syncthreads();
    if (warp == 1) tmem_dealloc(tmem_base, S::TMEM_COLS);
    return;
  }

  if (warp == 0) {
    // lane 0 streams the Q tiles and the K tiles, lane 1 the V tiles
    if (lane < 2) {
      const bool kside = lane == 0;
      const CUtensorMap* tm = kside ? &tmK : &tmV;
      uint8_t* ring = kside ? sK : sV;
      uint64_t* full = kside ? k_full : v_full;
      uint64_t* empty = kside ? k_empty : v_empty;
      asm volatile("prefetch.tensormap [%0];" ::"l"((uint64_t)tm) : "memory");
      if (kside) asm volatile("prefetch.tensormap [%0];" ::"l"((uint64_t)&tmQ) : "memory");
      const int nst = kside ? S::KST : 2;
      uint32_t armed[S::KST] = {}, q_armed[2] = {0, 0};
      SegIter it(use_sk, U, items, KT, blockIdx.x, gridDim.x);
      int item, kt0, kt1;
      int g = 0, si = 0;
      bool ok = true;
      while (ok && it.next(item, kt0, kt1)) {
        const int bh = item / QT, sq = bh / H, hq = bh % H;
        if (kside) {
          const int qb = si & 1;
          if (!mbar_wait(su32(&q_empty[qb]), ((si >> 1) & 1) ^ 1, abort_flag, err, 10)) break;
          mbar_expect_tx(su32(&q_full[qb]), S::Q_BYTES);
          const int q0 = (item % QT) * AT_BM;
          for (int b = 0; b < NB; ++b)
            tma_load_rows(su32(sQ + qb * S::Q_BYTES + b * AT_BM * 128), &tmQ, q_tok, b * 64, q0, hq,
                          sq, su32(&q_full[qb]));
          ++q_armed[qb];
        }
        for (int kt = kt0; kt < kt1; ++kt, ++g) {
          const int st = g % nst;
          if (!mbar_wait(su32(&empty[st]), ((g / nst) & 1) ^ 1, abort_flag, err, 11)) {
            ok = false;
            break;
          }
          mbar_expect_tx(su32(&full[st]), S::KV_BYTES);
          for (int b = 0; b < NB; ++b)
            tma_load_rows(su32(ring + st * S::KV_BYTES + b * AT_BN * 128), tm, kv_tok, b * 64,
                          kt * AT_BN, hq, sq, su32(&full[st]));
          ++armed[st];
        }
        ++si;
      }
      // Every copy this thread issued has landed before the CTA may exit.
      for (int i = 0; i < nst; ++i)
        if (armed[i] != 0) mbar_drain(su32(&full[i]), (armed[i] - 1) & 1, err, 15);
      for (int i = 0; i < 2; ++i)
        if (q_armed[i] != 0) mbar_drain(su32(&q_full[i]), (q_armed[i] - 1) & 1, err, 15);
    }
  } else if (warp == 1) {
    if (lane == 0) {
      constexpr uint32_t idS = idesc_bf16(AT_BM, AT_BN);
      constexpr uint32_t idO = idesc_bf16_bmn(AT_BM, HD);
      // Descriptors formed once, slices by offset (see k_attn_pp).
      const uint64_t dq0 = sdesc_sw128(su32(sQ)), dk0 = sdesc_sw128(su32(sK));
      const uint64_t dv0 = sdesc_sw128_mn(su32(sV), AT_BN * 128);
      // S(g) = Q K(g)^T for key tile g of segment si (q buffer si & 1).
      auto issue_s = [&](int g, int si, bool first, bool last) -> bool {
        const int qb = si & 1;
        if (first && !mbar_wait(su32(&q_full[qb]), (si >> 1) & 1, abort_flag, err, 13))
          return false;
        const int st = g % S::KST;
        if (!mbar_wait(su32(&k_full[st]), (g / S::KST) & 1, abort_flag, err, 12)) return false;
        tc_fence_after();
        const uint64_t qd = sdesc_add(dq0, qb * S::Q_BYTES), kd = sdesc_add(dk0, st * S::KV_BYTES);
        const uint32_t d = tmem_base + S::TM_S0 + (uint32_t)((g & 1) * AT_BN);
#pragma unroll
        for (int kk = 0; kk < HD / 16; ++kk)
          mma_bf16(d, sdesc_add(qd, (kk >> 2) * (AT_BM * 128) + (kk & 3) * 32),
                   sdesc_add(kd, (kk >> 2) * (AT_BN * 128) + (kk & 3) * 32), idS,
                   kk > 0 ? 1u : 0u);
        mma_commit(su32(&s_full[g & 1]));
        mma_commit(su32(&k_empty[st]));
        if (last) mma_commit(su32(&q_empty[qb]));
        return true;
      };
      // O(si & 1) += P(g) V(g) for key tile g of segment si.
      auto issue_pv = [&](int g, int si, bool first, bool last) -> bool {
        const int ob = si & 1, st = g & 1;
        if (first && !mbar_wait(su32(&o_empty[ob]), ((si >> 1) & 1) ^ 1, abort_flag, err, 20))
          return false;
        if (!mbar_wait(su32(&v_full[st]), (g >> 1) & 1, abort_flag, err, 21)) return false;
        if (!mbar_wait(su32(&p_full[g & 1]), (g >> 1) & 1, abort_flag, err, 14)) return false;
        tc_fence_after();
        const uint64_t vd = sdesc_add(dv0, st * S::KV_BYTES);
        // P keys 16kk..16kk+15: half kk/4 of the tile, columns 8(kk%4).. of that half's S
        const uint32_t pt = tmem_base + S::TM_S0 + (uint32_t)((g & 1) * AT_BN);
#pragma unroll
        for (int kk = 0; kk < AT_BN / 16; ++kk)
          mma_bf16_ts(tmem_base + (uint32_t)(ob * HD),
                      pt + (uint32_t)((kk >> 2) * (AT_BN / 2) + (kk & 3) * 8),
                      sdesc_add(vd, kk * 16 * 128), idO, (!first || kk > 0) ? 1u : 0u);
        mma_commit(su32(&v_empty[st]));
        mma_commit(su32(o_done));
        if (last) mma_commit(su32(&o_full[ob]));
        return true;
      };
      // Segments walked with one of lookahead: S of the next key tile (possibly
      // the next segment's first) is issued before P V of the current one.
      SegIter it(use_sk, U, items, KT, blockIdx.x, gridDim.x);
      int cur_item, c0, c1, nxt_item, n0 = 0, n1 = 0;
      bool have = it.next(cur_item, c0, c1);
      bool have_next = have && it.next(nxt_item, n0, n1);
      int g = 0, si = 0;
      bool ok = !have || issue_s(0, 0, true, c0 + 1 == c1);
      while (ok && have) {
        for (int kt = c0; kt < c1; ++kt, ++g) {
          if (kt + 1 < c1) {
            if (!issue_s(g + 1, si, false, kt + 2 == c1)) { ok = false; break; }
          } else if (have_next) {
            if (!issue_s(g + 1, si + 1, true, n0 + 1 == n1)) { ok = false; break; }
          }
          if (!issue_pv(g, si, kt == c0, kt + 1 == c1)) { ok = false; break; }
        }
        have = have_next;
        c0 = n0;
        c1 = n1;
        ++si;
        if (have) have_next = it.next(nxt_item, n0, n1);
      }
      (void)cur_item;
      // Every MMA this thread issued has completed before TMEM is freed.
      mma_commit(su32(done));
      mbar_drain(su32(done), 0, err, 16);
    }
  } else {
    // Softmax: warps 2-5 take keys 0-63 of each tile (and output columns
    // 0..HD/2), warps 6-9 keys 64-127 (and the other columns); one thread per
    // query row each.
    const int half = (warp - 2) >> 2;
    const int quarter = warp & 3;
    const int row = quarter * 32 + lane;
    const int wi = warp - 2;  // this warp's index among the softmax warps
    const uint32_t lane_off = (uint32_t)(quarter * 32) << 16;
    SegIter it(use_sk, U, items, KT, blockIdx.x, gridDim.x);
    int item, kt0, kt1;
    // key tiles, segments and exchange rounds (row maxima per tile, row sums
    // per segment) so far
    int g = 0, si = 0, e = 0;
    bool ok = true;
    while (ok && it.next(item, kt0, kt1)) {
      const int ob = si & 1;
      const uint32_t tO = tmem_base + lane_off + (uint32_t)(ob * HD + half * (HD / 2));
      float m = -INFINITY, l = 0.f;
      for (int kt = kt0; kt < kt1; ++kt, ++g, ++e) {
        const int sb = g & 1;
        if (!warp_wait(su32(&s_full[sb]), (g >> 1) & 1, abort_flag, err, 17)) {
          ok = false;
          break;
        }
        tc_fence_after();
        const uint32_t tS =
            tmem_base + lane_off + S::TM_S0 + (uint32_t)(sb * AT_BN) + (uint32_t)(half * AT_KH);
        const int kbase = kt * AT_BN + half * AT_KH;
        const bool full = kbase + AT_KH <= Lk;  // no key of this half-tile is past Lk
        uint32_t sv[AT_KH];                      // this row of S, this half of the tile
        tmem_ld32_nowait(tS, sv);
        tmem_ld32_nowait(tS + 32, sv + 32);
        tmem_ld_wait();
        if (!full) {
#pragma unroll
          for (int i = 0; i < AT_KH; ++i)
            if (kbase + i >= Lk) sv[i] = __float_as_uint(-INFINITY);
        }
        float pm[8];
#pragma unroll
        for (int j = 0; j < 8; ++j) pm[j] = __uint_as_float(sv[j]);
#pragma unroll
        for (int i = 8; i < AT_KH; ++i) pm[i & 7] = fmaxf(pm[i & 7], __uint_as_float(sv[i]));
        const float hmax = fmaxf(fmaxf(fmaxf(pm[0], pm[1]), fmaxf(pm[2], pm[3])),
                                 fmaxf(fmaxf(pm[4], pm[5]), fmaxf(pm[6], pm[7])));
        // exchange the half-row maxima with the other warpgroup
        float* xp = xch + (e & 1) * 2 * AT_BM;
        xp[half * AT_BM + row] = hmax;
        __syncwarp();
        if (lane == 0) mbar_arrive(su32(&xbar[e & 1]));
        if (!warp_wait(su32(&xbar[e & 1]), (e >> 1) & 1, abort_flag, err, 22)) {
          ok = false;
          break;
        }
        // finite: the first key of every key tile is valid
        const float mt = fmaxf(hmax, xp[(half ^ 1) * AT_BM + row]) * scale_log2;
        if (kt > kt0) {
          const bool need = mt > m + 8.f;
          if (__any_sync(0xffffffffu, need)) {
            // P V of the previous tile must be complete before O is rescaled.  That
            // of tile g-2 has completed (S(g) was issued after it), and that of
            // tile g needs this warp's P, so the parity names tile g-1.
            if (!warp_wait(su32(o_done), (g - 1) & 1, abort_flag, err, 18)) {
              ok = false;
              break;
            }
            tc_fence_after();
            const float alpha = need ? exp2_approx(m - mt) : 1.f;
            if (need) {
              m = mt;
              l *= alpha;
            }
            uint32_t r[32];
#pragma unroll 1
            for (int cc = 0; cc < HD / 64; ++cc) {
              tmem_ld32(tO + cc * 32, r);
#pragma unroll
              for (int i = 0; i < 32; ++i) r[i] = __float_as_uint(__uint_as_float(r[i]) * alpha);
              tmem_st32(tO + cc * 32, r);
            }
          }
        } else {
          m = mt;
        }
        // P = exp2(S * scale - m) for this half, two keys per TMEM column (the
        // lower key in the low 16 bits), over this half's first 32 S columns.
        float ps[8] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
        const float nm = -m;
        uint32_t pk[AT_KH / 2];
#pragma unroll
        for (int i = 0; i < AT_KH / 2; ++i) {
          const float p0 = exp2_approx(fmaf(__uint_as_float(sv[2 * i]), scale_log2, nm));
          const float p1 = exp2_approx(fmaf(__uint_as_float(sv[2 * i + 1]), scale_log2, nm));
          ps[(2 * i) & 7] += p0;
          ps[(2 * i + 1) & 7] += p1;
          pk[i] = pack_bf16x2(p0, p1);
        }
        tmem_st32(tS, pk);
        l += ((ps[0] + ps[1]) + (ps[2] + ps[3])) + ((ps[4] + ps[5]) + (ps[6] + ps[7]));
        tmem_st_wait();
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(su32(&p_full[sb]));
      }
      if (!ok) break;
      // End of the segment: combine the two groups' row sums, then read this
      // group's half of O once every P V of the segment has completed.
      float* xp = xch + (e & 1) * 2 * AT_BM;
      xp[half * AT_BM + row] = l;
      __syncwarp();
      if (lane == 0) mbar_arrive(su32(&xbar[e & 1]));
      if (!warp_wait(su32(&xbar[e & 1]), (e >> 1) & 1, abort_flag, err, 23)) break;
      const float lt = l + xp[(half ^ 1) * AT_BM + row];
      ++e;
      if (!warp_wait(su32(&o_full[ob]), (si >> 1) & 1, abort_flag, err, 19)) break;
      tc_fence_after();
      if (!segment_output<HD>(tO, m, lt, item, kt0, kt1, KT, QT, H, Lq, U, O, half, row, lane,
                              wi, sk, err, abort_flag))
        break;
      // This O buffer may now take the segment after next.
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(su32(&o_empty[ob]));
      ++si;
    }
  }

  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  if (warp == 1) {
    __syncwarp();
    tmem_dealloc(tmem_base, S::TMEM_COLS);
  }
}

// ---------------------------------------------------------------- two query tiles per item
// The default kernel.  An item is a pair of query tiles (256 query rows) of one
// (sequence, head); both tiles share every K and V tile the CTA loads.  Each
// tile has its own softmax warpgroup, one thread per query row holding the
// whole 128-key row of S, so no row statistics cross warpgroups.  The MMA
// warp interleaves the two tiles,
//   S0(j) S1(j) | PV0(j) S0(j+1) | PV1(j) S1(j+1) | PV0(j+1) ...
// so the tensor cores compute one tile's P V and next S while the other
// tile's softmax runs; P overwrites the first 64 columns of its tile's S
// buffer, and S(j+1) of a tile is issued after P V(j) of the same tile has
// been issued (tensor-core operations of one thread run in order).  With one
// S buffer and one O accumulator per tile TMEM holds 2 x (HD + 128) columns.
// Schedules, the stream-K combine and the bounded waits are those of the
// one-tile kernel above, with items of 256 rows.
constexpr int PP_THREADS = 320;  // warp 0 TMA, warp 1 MMA, warps 2-5 / 6-9 softmax of tile 0 / 1
// Of every 8 key pairs of a row, this many take their exponentials on the FMA
// pipe (exp2_poly_x2) instead of the special-function unit.
#ifndef ATTN_POLY_PAIRS
#define ATTN_POLY_PAIRS 0
#endif

template <int HD>
struct PpShape {
  static constexpr uint32_t QT_BYTES = AT_BM * HD * 2;  // one query tile
  static constexpr uint32_t KV_BYTES = AT_BN * HD * 2;  // one K or V tile
  static constexpr int KST = 3, VST = 2;                // K and V ring stages
  static constexpr size_t SMEM = 2 * QT_BYTES + (KST + VST) * (size_t)KV_BYTES + 256;
  // TMEM columns: O of tile t at t * HD, S (then P) of tile t at TM_S0 + 128 t
  static constexpr uint32_t TM_S0 = 2 * HD;
  static constexpr uint32_t TMEM_COLS = 512;
  static_assert(TM_S0 + 2 * AT_BN <= TMEM_COLS, "TMEM budget");
  // Stream-K slot: per softmax warp wi its 32 rows x HD columns of O (float4
  // index (wi * HD / 4 + c) * 32 + lane), then per warp m[32] and l[32].
  static constexpr int SLOT = 2 * AT_BM * HD + 8 * 2 * 32;
};

// Output of one query tile of a segment by one softmax warp (its 32 rows, all
// HD columns); see segment_output for the stream-K publish / combine.
template <int HD>
__device__ __forceinline__ bool segment_output_pp(uint32_t tO, float m, float lt, int item, int kt0,
                                                  int kt1, int KT, int QP, int H, int Lq,
                                                  int64_t U, bf16* __restrict__ O, int t, int row,
                                                  int lane, int wi, const AtSk& sk, int* err,
                                                  volatile int* abort_flag) {
  using S = PpShape<HD>;
  auto store32 = [&](bf16* dst, const float (&v)[32], float inv) {
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      uint4 u;
      u.x = pack_bf16x2(v[8 * j] * inv, v[8 * j + 1] * inv);
      u.y = pack_bf16x2(v[8 * j + 2] * inv, v[8 * j + 3] * inv);
      u.z = pack_bf16x2(v[8 * j + 4] * inv, v[8 * j + 5] * inv);
      u.w = pack_bf16x2(v[8 * j + 6] * inv, v[8 * j + 7] * inv);
      *reinterpret_cast<uint4*>(dst + 8 * j) = u;
    }
  };
  const int bh = item / QP, sq = bh / H, hq = bh % H;
  const int qrow = (item % QP) * (2 * AT_BM) + t * AT_BM + row;
  bf16* orow = O + (((int64_t)sq * Lq + qrow) * H + hq) * HD;
  if (kt0 == 0 && kt1 == KT) {
    const float inv = 1.f / lt;
#pragma unroll 1
    for (int cc = 0; cc < HD / 32; ++cc) {
      uint32_t r[32];
      tmem_ld32(tO + cc * 32, r);
      float v[32];
#pragma unroll
      for (int x = 0; x < 32; ++x) v[x] = __uint_as_float(r[x]);
      if (qrow < Lq) store32(orow + cc * 32, v, inv);
    }
    return true;
  }
  const int64_t iu = (int64_t)item * KT;
  const int w_first = sk_worker_of(iu, U, gridDim.x);
  const int nparts = sk_worker_of(iu + KT - 1, U, gridDim.x) - w_first + 1;
  const int part = (int)blockIdx.x - w_first;
  if (nparts > AT_MAX_PARTS) {  // excluded by the host's choice of schedule
    if (lane == 0) {
      *abort_flag = 1;
      atomicExch(err, 24);
    }
    return false;
  }
  auto slot_of = [&](int i) -> float* {
    const int wk = w_first + i;
    const int first_item = (int)(((int64_t)wk * U / gridDim.x) / KT);
    return sk.ws + (size_t)(2 * wk + (first_item == item ? 0 : 1)) * S::SLOT;
  };
  int* cnt = sk.cnt + 8 * item + wi;
  int last = 0;
  if (lane == 0) last = ld_acquire(cnt) == nparts - 1 ? 1 : 0;
  last = __shfl_sync(0xffffffffu, last, 0);
  if (!last) {
    float* mine = slot_of(part);
    float4* o4 = reinterpret_cast<float4*>(mine) + (size_t)wi * (HD / 4) * 32 + lane;
#pragma unroll 1
    for (int cc = 0; cc < HD / 32; ++cc) {
      uint32_t r[32];
      tmem_ld32(tO + cc * 32, r);
#pragma unroll
      for (int j = 0; j < 8; ++j)
        o4[(cc * 8 + j) * 32] =
            make_float4(__uint_as_float(r[4 * j]), __uint_as_float(r[4 * j + 1]),
                        __uint_as_float(r[4 * j + 2]), __uint_as_float(r[4 * j + 3]));
    }
    float* ml = mine + 2 * AT_BM * HD + wi * 64;
    ml[lane] = m;
    ml[32 + lane] = lt;
    __threadfence();
    __syncwarp();
    if (lane == 0) last = atomicAdd(cnt, 1) == nparts - 1 ? 1 : 0;
    last = __shfl_sync(0xffffffffu, last, 0);
  }
  if (last) {
    __threadfence();
    if (lane == 0) *cnt = 0;
    float wp[AT_MAX_PARTS], lp[AT_MAX_PARTS];
    float M = m;
#pragma unroll
    for (int i = 0; i < AT_MAX_PARTS; ++i) {
      wp[i] = -INFINITY;
      lp[i] = 0.f;
      if (i < nparts) {
        if (i == part) {
          wp[i] = m;
          lp[i] = lt;
        } else {
          const float* ml = slot_of(i) + 2 * AT_BM * HD + wi * 64;
          wp[i] = __ldcg(ml + lane);
          lp[i] = __ldcg(ml + 32 + lane);
        }
        M = fmaxf(M, wp[i]);
      }
    }
    float den = 0.f;
#pragma unroll
    for (int i = 0; i < AT_MAX_PARTS; ++i) {
      wp[i] = i < nparts ? exp2_approx(wp[i] - M) : 0.f;
      den = fmaf(wp[i], lp[i], den);
    }
    const float inv = 1.f / den;
#pragma unroll 1
    for (int cc = 0; cc < HD / 32; ++cc) {
      uint32_t r[32];
      tmem_ld32(tO + cc * 32, r);
      float acc[32];
#pragma unroll
      for (int x = 0; x < 32; ++x) acc[x] = 0.f;
#pragma unroll
      for (int i = 0; i < AT_MAX_PARTS; ++i) {
        if (i >= nparts) break;
        float xv[32];
        if (i == part) {
#pragma unroll
          for (int x = 0; x < 32; ++x) xv[x] = __uint_as_float(r[x]);
        } else {
          const float4* src =
              reinterpret_cast<const float4*>(slot_of(i)) + (size_t)wi * (HD / 4) * 32 + lane;
#pragma unroll
          for (int j = 0; j < 8; ++j) {
            const float4 q = __ldcg(src + (cc * 8 + j) * 32);
            xv[4 * j] = q.x; xv[4 * j + 1] = q.y; xv[4 * j + 2] = q.z; xv[4 * j + 3] = q.w;
          }
        }
#pragma unroll
        for (int x = 0; x < 32; ++x) acc[x] = fmaf(wp[i], xv[x], acc[x]);
      }
      if (qrow < Lq) store32(orow + cc * 32, acc, inv);
    }
  }
  return true;
}

template <int HD>
__global__ void __launch_bounds__(PP_THREADS, 1)
    k_attn_pp(const __grid_constant__ CUtensorMap tmQ, const __grid_constant__ CUtensorMap tmK,
              const __grid_constant__ CUtensorMap tmV, bf16* __restrict__ O, int H, int Lq, int Lk,
              float scale_log2, int q_tok, int kv_tok, int* err, int items, const AtSk sk) {
  using S = PpShape<HD>;
  constexpr int NB = HD / 64;  // 64-column boxes per row of Q/K/V
  extern __shared__ __align__(1024) uint8_t smem_raw[];
  uint8_t* smem = smem_raw;
  uint8_t* sQ = smem;                         // [2] query tiles of the item
  uint8_t* sK = sQ + 2 * S::QT_BYTES;         // [KST] K stages
  uint8_t* sV = sK + S::KST * S::KV_BYTES;    // [VST] V stages
  uint64_t* bars = (uint64_t*)(sV + S::VST * S::KV_BYTES);
  uint64_t* q_full = bars;        // both query tiles of the segment landed
  uint64_t* q_empty = bars + 1;   // the segment's last S MMAs completed
  uint64_t* k_full = bars + 2;    // [KST]
  uint64_t* k_empty = bars + 5;   // [KST] both S MMAs of the key tile completed
  uint64_t* v_full = bars + 8;    // [VST]
  uint64_t* v_empty = bars + 10;  // [VST] both P V MMAs of the key tile completed
  uint64_t* s_full = bars + 12;   // [2] per query tile: S of its current key tile
  uint64_t* p_full = bars + 14;   // [2] per query tile: P written (4 warps)
  uint64_t* o_full = bars + 16;   // [2] per query tile: every P V of the segment completed
  uint64_t* o_empty = bars + 18;  // [2] per query tile: the segment's O read out (4 warps)
  uint64_t* done = bars + 20;     // every MMA of the CTA has completed
  uint32_t* tmem_slot = (uint32_t*)(bars + 21);
  volatile int* abort_flag = (volatile int*)(tmem_slot + 1);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int QT = (Lq + AT_BM - 1) / AT_BM, KT = (Lk + AT_BN - 1) / AT_BN;
  const int QP = (QT + 1) / 2;  // query tile pairs per (sequence, head)
  const bool use_sk = sk.cnt != nullptr;
  const int64_t U = use_sk ? sk.units : (int64_t)items * KT;

  if (threadIdx.x == 0) {
    mbar_init(su32(q_full), 1);
    mbar_init(su32(q_empty), 1);
    for (int i = 0; i < S::KST; ++i) {
      mbar_init(su32(&k_full[i]), 1);
      mbar_init(su32(&k_empty[i]), 1);
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(su32(&v_full[i]), 1);
      mbar_init(su32(&v_empty[i]), 1);
      mbar_init(su32(&s_full[i]), 1);
      mbar_init(su32(&p_full[i]), 4);
      mbar_init(su32(&o_full[i]), 1);
      mbar_init(su32(&o_empty[i]), 4);
    }
    mbar_init(su32(done), 1);
    *abort_flag = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  if (warp == 1) tmem_alloc(su32(tmem_slot), S::TMEM_COLS);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem_base = *tmem_slot;
  pdl_wait();
  pdl_release();
  if ((su32(smem) & 1023u) != 0) {  // the 128-byte-swizzled tiles need 1024-byte alignment
    if (threadIdx.x == 0) atomicExch(err, 25);
    __syncthreads();
    if (warp == 1) tmem_dealloc(tmem_base, S::TMEM_COLS);
    return;
  }

  if (warp == 0) {
    // lane 0 streams the query tile pairs and the K tiles, lane 1 the V tiles
    if (lane < 2) {
      const bool kside = lane == 0;
      const CUtensorMap* tm = kside ? &tmK : &tmV;
      uint8_t* ring = kside ? sK : sV;
      uint64_t* full = kside ? k_full : v_full;
      uint64_t* empty = kside ? k_empty : v_empty;
      asm volatile("prefetch.tensormap [%0];" ::"l"((uint64_t)tm) : "memory");
      if (kside) asm volatile("prefetch.tensormap [%0];" ::"l"((uint64_t)&tmQ) : "memory");
      const int nst = kside ? S::KST : S::VST;
      uint32_t armed[S::KST] = {}, q_armed = 0;
      SegIter it(use_sk, U, items, KT, blockIdx.x, gridDim.x);
      int item, kt0, kt1;
      int g = 0, si = 0;
      bool ok = true;
      while (ok && it.next(item, kt0, kt1)) {
        const int bh = item / QP, sq = bh / H, hq = bh % H;
        if (kside) {
          if (!mbar_wait(su32(q_empty), (si & 1) ^ 1, abort_flag, err, 10)) break;
          mbar_expect_tx(su32(q_full), 2 * S::QT_BYTES);
          const int q0 = (item % QP) * (2 * AT_BM);
          for (int t = 0; t < 2; ++t)
            for (int b = 0; b < NB; ++b)
              tma_load_rows(su32(sQ + t * S::QT_BYTES + b * AT_BM * 128), &tmQ, q_tok, b * 64,
                            q0 + t * AT_BM, hq, sq, su32(q_full));
          ++q_armed;
        }
        for (int kt = kt0; kt < kt1; ++kt, ++g) {
          const int st = g % nst;
          if (!mbar_wait(su32(&empty[st]), ((g / nst) & 1) ^ 1, abort_flag, err, 11)) {
            ok = false;
            break;
          }
          mbar_expect_tx(su32(&full[st]), S::KV_BYTES);
          for (int b = 0; b < NB; ++b)
            tma_load_rows(su32(ring + st * S::KV_BYTES + b * AT_BN * 128), tm, kv_tok, b * 64,
                          kt * AT_BN, hq, sq, su32(&full[st]));
          ++armed[st];
        }
        ++si;
      }
      for (int i = 0; i < nst; ++i)
        if (armed[i] != 0) mbar_drain(su32(&full[i]), (armed[i] - 1) & 1, err, 15);
      if (q_armed != 0) mbar_drain(su32(q_full), (q_armed - 1) & 1, err, 15);
    }
  } else if (warp == 1) {
    if (lane == 0) {
      constexpr uint32_t idS = idesc_bf16(AT_BM, AT_BN);
      constexpr uint32_t idO = idesc_bf16_bmn(AT_BM, HD);
      // Shared-memory descriptors are formed once: a 16-column slice's
      // descriptor is its tile's plus the slice's byte offset / 16 in the
      // start-address field (see sdesc_add).  Issuing a group of 16 MMAs this
      // way instead of building each descriptor from its address took the 14B
      // self-attention from 32.6 to 31.9 ms: the MMA thread's issue sits on the
      // softmax -> P V -> S chain.
      const uint64_t dq0 = sdesc_sw128(su32(sQ)), dk0 = sdesc_sw128(su32(sK));
      const uint64_t dv0 = sdesc_sw128_mn(su32(sV), AT_BN * 128);
      // S_t = Q_t K(g)^T into tile t's S buffer (K stage already waited for).
      auto issue_s = [&](int t, int g) {
        const uint64_t qd = sdesc_add(dq0, t * S::QT_BYTES);
        const uint64_t kd = sdesc_add(dk0, (g % S::KST) * S::KV_BYTES);
        const uint32_t d = tmem_base + S::TM_S0 + (uint32_t)(t * AT_BN);
#pragma unroll
        for (int kk = 0; kk < HD / 16; ++kk)
          mma_bf16(d, sdesc_add(qd, (kk >> 2) * (AT_BM * 128) + (kk & 3) * 32),
                   sdesc_add(kd, (kk >> 2) * (AT_BN * 128) + (kk & 3) * 32), idS,
                   kk > 0 ? 1u : 0u);
        mma_commit(su32(&s_full[t]));
      };
      // O_t (+)= P_t(g) V(g); P keys 16kk..16kk+15 sit in S columns 8kk..8kk+7.
      auto issue_pv = [&](int t, int g, bool first) {
        const uint64_t vd = sdesc_add(dv0, (g % S::VST) * S::KV_BYTES);
        const uint32_t pt = tmem_base + S::TM_S0 + (uint32_t)(t * AT_BN);
#pragma unroll
        for (int kk = 0; kk < AT_BN / 16; ++kk)
          mma_bf16_ts(tmem_base + (uint32_t)(t * HD), pt + (uint32_t)(kk * 8),
                      sdesc_add(vd, kk * 16 * 128), idO, (!first || kk > 0) ? 1u : 0u);
      };
      SegIter it(use_sk, U, items, KT, blockIdx.x, gridDim.x);
      int item, c0, c1;
      int g = 0, si = 0;  // key tiles and segments so far
      bool ok = true;
      while (ok && it.next(item, c0, c1)) {
        const int n = c1 - c0;
        if (!mbar_wait(su32(q_full), si & 1, abort_flag, err, 13)) break;
        {
          const int st = g % S::KST;
          if (!mbar_wait(su32(&k_full[st]), (g / S::KST) & 1, abort_flag, err, 12)) break;
          tc_fence_after();
          issue_s(0, g);
          issue_s(1, g);
          mma_commit(su32(&k_empty[st]));
          if (n == 1) mma_commit(su32(q_empty));
        }
        for (int j = 1; j <= n; ++j) {
          const int gp = g + j - 1;  // the key tile whose P V is issued now
          const int gn = g + j;      // the key tile whose S is issued now (j < n)
          const int vst = gp % S::VST;
          if (!mbar_wait(su32(&v_full[vst]), (gp / S::VST) & 1, abort_flag, err, 21)) {
            ok = false;
            break;
          }
          // query tile 0: P V of tile gp, then S of tile gn
          if (j == 1 && !mbar_wait(su32(&o_empty[0]), (si & 1) ^ 1, abort_flag, err, 20)) {
            ok = false;
            break;
          }
          if (!mbar_wait(su32(&p_full[0]), gp & 1, abort_flag, err, 14)) {
            ok = false;
            break;
          }
          tc_fence_after();
          issue_pv(0, gp, j == 1);
          if (j == n) mma_commit(su32(&o_full[0]));
          if (j < n) {
            const int kst = gn % S::KST;
            if (!mbar_wait(su32(&k_full[kst]), (gn / S::KST) & 1, abort_flag, err, 12)) {
              ok = false;
              break;
            }
            tc_fence_after();
            issue_s(0, gn);
          }
          // query tile 1
          if (j == 1 && !mbar_wait(su32(&o_empty[1]), (si & 1) ^ 1, abort_flag, err, 20)) {
            ok = false;
            break;
          }
          if (!mbar_wait(su32(&p_full[1]), gp & 1, abort_flag, err, 14)) {
            ok = false;
            break;
          }
          tc_fence_after();
          issue_pv(1, gp, j == 1);
          mma_commit(su32(&v_empty[vst]));
          if (j == n) mma_commit(su32(&o_full[1]));
          if (j < n) {
            issue_s(1, gn);
            mma_commit(su32(&k_empty[gn % S::KST]));
            if (j == n - 1) mma_commit(su32(q_empty));
          }
        }
        g += n;
        ++si;
      }
      mma_commit(su32(done));
      mbar_drain(su32(done), 0, err, 16);
    }
  } else {
    // Softmax of query tile t: one thread per row (TMEM lane), all 128 keys.
    const int t = (warp - 2) >> 2;
    const int quarter = warp & 3;
    const int row = quarter * 32 + lane;
    const int wi = warp - 2;
    const uint32_t lane_off = (uint32_t)(quarter * 32) << 16;
    const uint32_t tO = tmem_base + lane_off + (uint32_t)(t * HD);
    const uint32_t tS = tmem_base + lane_off + S::TM_S0 + (uint32_t)(t * AT_BN);
    SegIter it(use_sk, U, items, KT, blockIdx.x, gridDim.x);
    int item, kt0, kt1;
    int g = 0, si = 0;
    bool ok = true;
    while (ok && it.next(item, kt0, kt1)) {
      float m = -INFINITY, l = 0.f;
      for (int kt = kt0; kt < kt1; ++kt, ++g) {
        if (!warp_wait(su32(&s_full[t]), g & 1, abort_flag, err, 17)) {
          ok = false;
          break;
        }
        tc_fence_after();
        uint32_t sv[AT_BN];
        tmem_ld32_nowait(tS, sv);
        tmem_ld32_nowait(tS + 32, sv + 32);
        tmem_ld32_nowait(tS + 64, sv + 64);
        tmem_ld32_nowait(tS + 96, sv + 96);
        tmem_ld_wait();
        const int kbase = kt * AT_BN;
        if (kbase + AT_BN > Lk) {
#pragma unroll
          for (int i = 0; i < AT_BN; ++i)
            if (kbase + i >= Lk) sv[i] = __float_as_uint(-INFINITY);
        }
        // Row maximum: eight running maxima, two new keys each per three-input max.
        float pm[8];
#pragma unroll
        for (int j = 0; j < 8; ++j) pm[j] = fmaxf(__uint_as_float(sv[j]), __uint_as_float(sv[8 + j]));
#pragma unroll
        for (int i = 16; i < AT_BN; i += 16) {
#pragma unroll
          for (int j = 0; j < 8; ++j)
            pm[j] = fmax3(pm[j], __uint_as_float(sv[i + j]), __uint_as_float(sv[i + 8 + j]));
        }
        const float rmax =
            fmaxf(fmax3(pm[0], pm[1], pm[2]), fmax3(fmax3(pm[3], pm[4], pm[5]), pm[6], pm[7]));
        // finite: the first key of every key tile is valid
        const float mt = rmax * scale_log2;
        // Lazy rescaling: the running maximum moves only when it grows by more
        // than 2^8; O is then rescaled below, after S is consumed.
        float alpha = 1.f;
        bool rescale = false;
        if (kt > kt0) {
          const bool need = mt > m + 8.f;
          rescale = __any_sync(0xffffffffu, need);
          if (need) {
            alpha = exp2_approx(m - mt);
            m = mt;
            l *= alpha;
          }
        } else {
          m = mt;
        }
        // P = exp2(S * scale - m), keys 16c..16c+15 packed into S columns 8c..8c+7.
        // The scale-and-shift and the row sum run as packed f32x2 operations on
        // key pairs (one instruction per pair), four running pair sums.
        const uint64_t sc2 = f32x2(scale_log2, scale_log2), nm2 = f32x2(-m, -m);
        uint64_t ps2[4];
#pragma unroll
        for (int c = 0; c < AT_BN / 16; ++c) {
          uint32_t pk[8];
#pragma unroll
          for (int i = 0; i < 8; ++i) {
            float x0, x1;
            f32x2_split(fma_f32x2(f32x2(__uint_as_float(sv[16 * c + 2 * i]),
                                        __uint_as_float(sv[16 * c + 2 * i + 1])),
                                  sc2, nm2),
                        x0, x1);
            float p0, p1;
            if (ATTN_POLY_PAIRS > 0 && (i & 7) >= 8 - ATTN_POLY_PAIRS) {
              f32x2_split(exp2_poly_x2(x0, x1), p0, p1);  // FMA pipe (see exp2_poly_x2)
            } else {
              p0 = exp2_approx(x0);
              p1 = exp2_approx(x1);
            }
            const uint64_t pp = f32x2(p0, p1);
            ps2[i & 3] = c == 0 && i < 4 ? pp : add_f32x2(ps2[i & 3], pp);
            pk[i] = pack_bf16x2(p0, p1);
          }
          tmem_st8(tS + 8 * c, pk);
        }
        {
          float a0, a1;
          f32x2_split(add_f32x2(add_f32x2(ps2[0], ps2[1]), add_f32x2(ps2[2], ps2[3])), a0, a1);
          l += a0 + a1;
        }
        if (rescale) {
          // O_t is idle: S_t of this key tile was issued after P V of the
          // previous one, whose completion the s_full wait observed; P V of
          // this tile waits for p_full below.
          uint32_t r[32];
#pragma unroll 1
          for (int cc = 0; cc < HD / 32; ++cc) {
            tmem_ld32(tO + cc * 32, r);
#pragma unroll
            for (int i = 0; i < 32; ++i) r[i] = __float_as_uint(__uint_as_float(r[i]) * alpha);
            tmem_st32(tO + cc * 32, r);
          }
        }
        tmem_st_wait();
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(su32(&p_full[t]));
      }
      if (!ok) break;
      if (!warp_wait(su32(&o_full[t]), si & 1, abort_flag, err, 19)) break;
      tc_fence_after();
      if (!segment_output_pp<HD>(tO, m, l, item, kt0, kt1, KT, QP, H, Lq, U, O, t, row, lane, wi,
                                 sk, err, abort_flag))
        break;
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(su32(&o_empty[t]));
      ++si;
    }
  }

  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  if (warp == 1) {
    __syncwarp();
    tmem_dealloc(tmem_base, S::TMEM_COLS);
  }
}

// 4-D tensor map of one operand, dimensions ordered by increasing stride:
// (hd, H, L, S) when token-major (hs < ls), (hd, L, H, S) when head-major;
// the box covers 64 columns of `rows` consecutive positions of one head.
bool make_tmap_op(CUtensorMap* tm, const AttnOperand& op, int hd, int L, int H, int S_,
                  uint32_t rows, int* tok) {
  EncodeTiledFn enc = encode_tiled_fn();
  if (enc == nullptr) return false;
  *tok = op.hs < op.ls ? 1 : 0;
  cuuint64_t dims[4], strides[3];
  cuuint32_t box[4];
  dims[0] = (cuuint64_t)hd;
  box[0] = 64;
  if (*tok) {
    dims[1] = (cuuint64_t)H; dims[2] = (cuuint64_t)L;
    strides[0] = (cuuint64_t)op.hs * 2; strides[1] = (cuuint64_t)op.ls * 2;
    box[1] = 1; box[2] = rows;
  } else {
    dims[1] = (cuuint64_t)L; dims[2] = (cuuint64_t)H;
    strides[0] = (cuuint64_t)op.ls * 2; strides[1] = (cuuint64_t)op.hs * 2;
    box[1] = rows; box[2] = 1;
  }
  dims[3] = (cuuint64_t)S_;
  strides[2] = (cuuint64_t)op.ss * 2;
  box[3] = 1;
  cuuint32_t estr[4] = {1, 1, 1, 1};
  return enc(tm, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 4, const_cast<void*>(op.ptr), dims, strides, box,
             estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
             CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

std::atomic<int> g_attn_schedule{0};

// Schedule by a makespan model in key-tile units: data-parallel costs
// ceil(items / G) x (KT + AT_OV), stream-K U / G + items / G x AT_OV + AT_FIX,
// where AT_OV is the per-item cost of loading Q and writing the output and
// AT_FIX the fix-up of a split item (publish, counter round trips, combine).
// Stream-K must win by 3 %: near-ties measured slower.
constexpr double AT_OV = 1.5, AT_FIX = 6.0;

template <int HD>
cudaError_t launch_attn_tc(const AttnOperand& Q, const AttnOperand& K, const AttnOperand& V,
                           void* O, int S_, int H, int Lq, int Lk, cudaStream_t s) {
  using S1 = AtShape<HD>;
  static_assert(S1::SMEM <= 232448, "shared memory budget");
  CUtensorMap tq, tk, tv;
  int q_tok = 0, k_tok = 0, v_tok = 0;
  if (!make_tmap_op(&tq, Q, HD, Lq, H, S_, AT_BM, &q_tok) ||
      !make_tmap_op(&tk, K, HD, Lk, H, S_, AT_BN, &k_tok) ||
      !make_tmap_op(&tv, V, HD, Lk, H, S_, AT_BN, &v_tok) || k_tok != v_tok)
    return cudaErrorInvalidValue;
  int* err = device_error_word();
  if (err == nullptr) return cudaErrorMemoryAllocation;
  const float scale_log2 = (float)(1.4426950408889634 / sqrt((double)HD));
  cudaError_t e = cudaFuncSetAttribute(k_attn_tc<HD>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       (int)S1::SMEM);
  if (e != cudaSuccess) return e;
  const int QT = (Lq + AT_BM - 1) / AT_BM, KT = (Lk + AT_BN - 1) / AT_BN;
  const int64_t items = (int64_t)S_ * H * QT;
  if (items > (1 << 26)) return cudaErrorInvalidValue;
  const int G = num_sms();
  int grid = items < G ? (int)items : G;
  AtSk sk = {nullptr, nullptr, 0};
  const int mode = g_attn_schedule.load() & 3;
  if (mode != 1) {
    const int64_t U = items * KT, per = U / G;
    const bool spans_ok = per > 0 && 1 + (KT - 1 + per - 1) / per <= AT_MAX_PARTS;
    const double dp_cost = (double)((items + G - 1) / G) * (KT + AT_OV);
    const double sk_cost = (double)U / G + (double)items / G * AT_OV + AT_FIX;
    if (spans_ok && (mode == 2 || sk_cost < 0.97 * dp_cost) &&
        sk_scratch(s, (size_t)8 * items, (size_t)2 * G * S1::SLOT, &sk.cnt, &sk.ws)) {
      sk.units = U;
      grid = G;
    } else {
      sk = {nullptr, nullptr, 0};
    }
  }
  count_launch();
  return launch_pdl(k_attn_tc<HD>, grid, AT_THREADS, S1::SMEM, s, tq, tk, tv, (bf16*)O, H, Lq, Lk,
                    scale_log2, q_tok, k_tok, err, (int)items, sk);
}

// The same model for the two-tile kernel, in units of one key tile for both
// query tiles of an item.
constexpr double PP_OV = 1.5, PP_FIX = 4.0;

template <int HD>
cudaError_t launch_attn_pp(const AttnOperand& Q, const AttnOperand& K, const AttnOperand& V,
                           void* O, int S_, int H, int Lq, int Lk, cudaStream_t s) {
  using S1 = PpShape<HD>;
  static_assert(S1::SMEM <= 232448, "shared memory budget");
  CUtensorMap tq, tk, tv;
  int q_tok = 0, k_tok = 0, v_tok = 0;
  if (!make_tmap_op(&tq, Q, HD, Lq, H, S_, AT_BM, &q_tok) ||
      !make_tmap_op(&tk, K, HD, Lk, H, S_, AT_BN, &k_tok) ||
      !make_tmap_op(&tv, V, HD, Lk, H, S_, AT_BN, &v_tok) || k_tok != v_tok)
    return cudaErrorInvalidValue;
  int* err = device_error_word();
  if (err == nullptr) return cudaErrorMemoryAllocation;
  const float scale_log2 = (float)(1.4426950408889634 / sqrt((double)HD));
  cudaError_t e = cudaFuncSetAttribute(k_attn_pp<HD>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       (int)S1::SMEM);
  if (e != cudaSuccess) return e;
  const int QT = (Lq + AT_BM - 1) / AT_BM, KT = (Lk + AT_BN - 1) / AT_BN;
  const int64_t items = (int64_t)S_ * H * ((QT + 1) / 2);
  if (items > (1 << 26)) return cudaErrorInvalidValue;
  const int G = num_sms();
  int grid = items < G ? (int)items : G;
  AtSk sk = {nullptr, nullptr, 0};
  const int mode = g_attn_schedule.load() & 3;
  if (mode != 1) {
    const int64_t U = items * KT, per = U / G;
    const bool spans_ok = per > 0 && 1 + (KT - 1 + per - 1) / per <= AT_MAX_PARTS;
    const double dp_cost = (double)((items + G - 1) / G) * (KT + PP_OV);
    const double sk_cost = (double)U / G + (double)items / G * PP_OV + PP_FIX;
    if (spans_ok && (mode == 2 || sk_cost < 0.97 * dp_cost) &&
        sk_scratch(s, (size_t)8 * items, (size_t)2 * G * S1::SLOT, &sk.cnt, &sk.ws)) {
      sk.units = U;
      grid = G;
    } else {
      sk = {nullptr, nullptr, 0};
    }
  }
  count_launch();
  return launch_pdl(k_attn_pp<HD>, grid, PP_THREADS, S1::SMEM, s, tq, tk, tv, (bf16*)O, H, Lq, Lk,
                    scale_log2, q_tok, k_tok, err, (int)items, sk);
}

}  // namespace

void set_attention_schedule(int mode) { g_attn_schedule.store(mode); }

cudaError_t attention_bf16(const AttnOperand& Q, const AttnOperand& K, const AttnOperand& V,
                           void* O, int S, int H, int Lq, int Lk, int hd, cudaStream_t s) {
  if (S <= 0 || Lq <= 0) return cudaSuccess;
  if (Lk <= 0) return cudaErrorInvalidValue;
  if ((((uintptr_t)Q.ptr) | ((uintptr_t)K.ptr) | ((uintptr_t)V.ptr) | ((uintptr_t)O)) & 15)
    return cudaErrorMisalignedAddress;
  // The one-tile kernel double-buffers Q, so it pays less per work item; it is
  // taken by default for short key ranges (cross-attention to 512 text tokens)
  // when the pair kernel would have at most two items per SM: there a work item
  // is a few key tiles and the pair kernel's exposed Q load dominates (measured
  // at one 3510-token sequence: 26 against 28 us).
  const int QT = (Lq + AT_BM - 1) / AT_BM, KT = (Lk + AT_BN - 1) / AT_BN;
  const int64_t pair_items = (int64_t)S * H * ((QT + 1) / 2);
  const bool one_tile = (g_attn_schedule.load() & 4) != 0 ||
                        (KT <= 4 && pair_items <= 2 * (int64_t)num_sms());
  if (hd == 128)
    return one_tile ? launch_attn_tc<128>(Q, K, V, O, S, H, Lq, Lk, s)
                    : launch_attn_pp<128>(Q, K, V, O, S, H, Lq, Lk, s);
  if (hd == 64)
    return one_tile ? launch_attn_tc<64>(Q, K, V, O, S, H, Lq, Lk, s)
                    : launch_attn_pp<64>(Q, K, V, O, S, H, Lq, Lk, s);
  return cudaErrorInvalidValue;
}

}  // namespace track
