// Flash attention on the sm_103a tensor cores (bf16 in, fp32 accumulate):
// O = softmax(Q K^T / sqrt(hd)) V per (sequence, head), no mask.
//
// One CTA per 128-query tile of one (sequence, head), 192 threads:
//   warp 0      TMA: the Q tile once, then K and V tiles of 128 keys, K through
//               a three-stage ring (lane 0) and V through a two-stage ring
//               (lane 1); 4-D tensor maps over head-major or token-major
//               operands, 128-byte swizzle, zero fill past L.  A K stage is
//               released as soon as S = Q K^T of its tile completes.
//   warp 1      allocates TMEM (O: hd columns; S: two 128-column buffers) and
//               issues, from one thread, S(j+1) = Q K(j+1)^T while the softmax
//               warps work on S(j), then O += P(j) V(j) once P(j) is ready.  P
//               is read from TMEM (the A operand of the MMA), V is the MN-major
//               B operand from shared memory, so no transposed copy is needed.
//   warps 2-9   softmax, two warpgroups splitting each 128-key tile by columns
//               (64 keys each), one thread per query row (its TMEM lane): row
//               maximum over the valid keys (halves combined through shared
//               memory), lazy rescaling of O (only when the running maximum
//               grows by more than 2^8; each group rescales its half of O's
//               columns in TMEM, after P V of the previous tile completes),
//               P = exp2(S * log2(e)/sqrt(hd) - m) rounded to bf16 pairs and
//               written over the first 32 of the group's 64 S columns, and at
//               the end O / l stored to the token-major output.  Because P
//               lives in the S buffer it came from, the softmax of tile j+1
//               never waits for P V of tile j unless it must rescale O.
// Tensor-core operations issued by one thread execute in issue order, so
// S(j+2), issued after O += P(j) V(j), overwrites P(j) only after it was read.
// Every mbarrier wait is bounded (see tc_common.cuh).
#include <cuda.h>
#include <cuda_bf16.h>
#include <math.h>

#include "internal.h"
#include "tc_common.cuh"

namespace track {

namespace {

using namespace tc;
typedef __nv_bfloat16 bf16;

constexpr int AT_BM = 128;       // query rows per CTA (MMA M)
constexpr int AT_BN = 128;       // keys per tile
constexpr int AT_THREADS = 320;  // warp 0 TMA, warp 1 MMA, warps 2-9 softmax
constexpr uint32_t TM_S0 = 128;  // TMEM column of S buffer 0 (buffer 1 at 256)

template <int HD>
struct AtShape {
  static constexpr uint32_t Q_BYTES = AT_BM * HD * 2;   // HD/64 boxes of [128 rows][128 B]
  static constexpr uint32_t KV_BYTES = AT_BN * HD * 2;  // one K or V tile
  static constexpr uint32_t X_BYTES = 2 * 2 * AT_BM * 4;  // row partials [parity][half][row]
  static constexpr int KST = 3;  // K ring stages
  static constexpr int VST = 2;  // V ring stages
  static constexpr size_t SMEM = 1024 + Q_BYTES + (KST + VST) * KV_BYTES + X_BYTES + 256;
  static constexpr uint32_t TMEM_COLS = 512;
};

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

template <int HD>
__global__ void __launch_bounds__(AT_THREADS, 1)
    k_attn_tc(const __grid_constant__ CUtensorMap tmQ, const __grid_constant__ CUtensorMap tmK,
              const __grid_constant__ CUtensorMap tmV, bf16* __restrict__ O, int H, int Lq, int Lk,
              float scale_log2, int q_tok, int kv_tok, int* err) {
  using S = AtShape<HD>;
  constexpr int NB = HD / 64;  // 64-column boxes per row of Q/K/V
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = (uint8_t*)(((uintptr_t)smem_raw + 1023) & ~(uintptr_t)1023);
  uint8_t* sQ = smem;
  uint8_t* sK = sQ + S::Q_BYTES;
  uint8_t* sV = sK + S::KST * S::KV_BYTES;
  float* xch = (float*)(sV + S::VST * S::KV_BYTES);  // [2][2][AT_BM] partial row maxima / sums
  uint64_t* bars = (uint64_t*)((uint8_t*)xch + S::X_BYTES);
  uint64_t* q_full = bars;
  uint64_t* k_full = bars + 1;    // [3] per K stage
  uint64_t* k_empty = bars + 4;   // [3] freed once S = Q K^T of the tile has completed
  uint64_t* v_full = bars + 7;    // [2] per V stage
  uint64_t* v_empty = bars + 9;   // [2] freed once P V of the tile has completed
  uint64_t* s_full = bars + 11;   // [2] per S buffer
  uint64_t* p_full = bars + 13;   // [2] P of the tile written into its S buffer (8 softmax warps)
  uint64_t* o_done = bars + 15;   // P V of the tile has completed
  uint64_t* xbar = bars + 16;     // [2] both halves' row partials written (per parity)
  uint64_t* done = bars + 18;     // every MMA of the CTA has completed
  uint32_t* tmem_slot = (uint32_t*)(bars + 19);
  volatile int* abort_flag = (volatile int*)(tmem_slot + 1);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int bh = blockIdx.y, q0 = blockIdx.x * AT_BM;
  const int sq = bh / H, hq = bh % H;
  const int nkt = (Lk + AT_BN - 1) / AT_BN;

  if (threadIdx.x == 0) {
    mbar_init(su32(q_full), 1);
    for (int i = 0; i < S::KST; ++i) {
      mbar_init(su32(&k_full[i]), 1);
      mbar_init(su32(&k_empty[i]), 1);
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(su32(&v_full[i]), 1);
      mbar_init(su32(&v_empty[i]), 1);
      mbar_init(su32(&s_full[i]), 1);
      mbar_init(su32(&p_full[i]), 8);
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

  if (warp == 0) {
    // lane 0 streams Q and the K tiles, lane 1 the V tiles, each through its own ring
    if (lane < 2) {
      const bool kside = lane == 0;
      const CUtensorMap* tm = kside ? &tmK : &tmV;
      uint8_t* ring = kside ? sK : sV;
      uint64_t* full = kside ? k_full : v_full;
      uint64_t* empty = kside ? k_empty : v_empty;
      asm volatile("prefetch.tensormap [%0];" ::"l"((uint64_t)tm) : "memory");
      if (kside) {
        asm volatile("prefetch.tensormap [%0];" ::"l"((uint64_t)&tmQ) : "memory");
        mbar_expect_tx(su32(q_full), S::Q_BYTES);
        for (int b = 0; b < NB; ++b)
          tma_load_rows(su32(sQ + b * AT_BM * 128), &tmQ, q_tok, b * 64, q0, hq, sq, su32(q_full));
      }
      const int nst = kside ? S::KST : S::VST;
      uint32_t armed[S::KST] = {};
      for (int kt = 0; kt < nkt; ++kt) {
        const int st = kt % nst;
        if (!mbar_wait(su32(&empty[st]), ((kt / nst) & 1) ^ 1, abort_flag, err, 11)) break;
        mbar_expect_tx(su32(&full[st]), S::KV_BYTES);
        for (int b = 0; b < NB; ++b)
          tma_load_rows(su32(ring + st * S::KV_BYTES + b * AT_BN * 128), tm, kv_tok, b * 64,
                        kt * AT_BN, hq, sq, su32(&full[st]));
        ++armed[st];
      }
      // Every copy this thread issued has landed before the CTA may exit.
      if (kside) mbar_drain(su32(q_full), 0, err, 15);
      for (int i = 0; i < nst; ++i)
        if (armed[i] != 0) mbar_drain(su32(&full[i]), (armed[i] - 1) & 1, err, 15);
    }
  } else if (warp == 1) {
    if (lane == 0) {
      constexpr uint32_t idS = idesc_bf16(AT_BM, AT_BN);
      constexpr uint32_t idO = idesc_bf16_bmn(AT_BM, HD);
      const uint32_t qa = su32(sQ);
      auto issue_s = [&](int kt) -> bool {
        const int st = kt % S::KST;
        if (!mbar_wait(su32(&k_full[st]), (kt / S::KST) & 1, abort_flag, err, 12)) return false;
        tc_fence_after();
        const uint32_t ka = su32(sK + st * S::KV_BYTES);
        const uint32_t d = tmem_base + TM_S0 + (uint32_t)((kt & 1) * AT_BN);
#pragma unroll
        for (int kk = 0; kk < HD / 16; ++kk)
          mma_bf16(d, sdesc_sw128(qa + (kk >> 2) * (AT_BM * 128) + (kk & 3) * 32),
                   sdesc_sw128(ka + (kk >> 2) * (AT_BN * 128) + (kk & 3) * 32), idS,
                   kk > 0 ? 1u : 0u);
        mma_commit(su32(&s_full[kt & 1]));
        mma_commit(su32(&k_empty[st]));
        return true;
      };
      bool ok = mbar_wait(su32(q_full), 0, abort_flag, err, 13);
      if (ok) {
        tc_fence_after();
        ok = issue_s(0);
      }
      for (int kt = 0; ok && kt < nkt; ++kt) {
        if (kt + 1 < nkt && !issue_s(kt + 1)) break;
        const int st = kt & 1;  // V stage and S/P buffer of this tile
        if (!mbar_wait(su32(&v_full[st]), (kt >> 1) & 1, abort_flag, err, 21)) break;
        if (!mbar_wait(su32(&p_full[st]), (kt >> 1) & 1, abort_flag, err, 14)) break;
        tc_fence_after();
        const uint32_t va = su32(sV + st * S::KV_BYTES);
        // P keys 16kk..16kk+15: half kk/4 of the tile, columns 8(kk%4).. of that half's S
        const uint32_t pt = tmem_base + TM_S0 + (uint32_t)(st * AT_BN);
#pragma unroll
        for (int kk = 0; kk < AT_BN / 16; ++kk)
          mma_bf16_ts(tmem_base, pt + (uint32_t)((kk >> 2) * (AT_BN / 2) + (kk & 3) * 8),
                      sdesc_sw128_mn(va + kk * 16 * 128, AT_BN * 128), idO,
                      (kt > 0 || kk > 0) ? 1u : 0u);
        mma_commit(su32(&v_empty[st]));
        mma_commit(su32(o_done));
      }
      // Every MMA this thread issued has completed before TMEM is freed.
      mma_commit(su32(done));
      mbar_drain(su32(done), 0, err, 16);
    }
  } else {
    // Softmax: warps 2-5 take keys 0-63 of each tile (and O columns 0..HD/2), warps
    // 6-9 keys 64-127 (and the other O columns); one thread per query row each.
    const int half = (warp - 2) >> 2;
    const int quarter = warp & 3;
    const int row = quarter * 32 + lane;
    const uint32_t lane_off = (uint32_t)(quarter * 32) << 16;
    const uint32_t tO = tmem_base + lane_off + (uint32_t)(half * (HD / 2));
    constexpr int KH = AT_BN / 2;  // keys per half
    float m = -INFINITY, l = 0.f;
    bool ok = true;
    for (int kt = 0; kt < nkt; ++kt) {
      if (!warp_wait(su32(&s_full[kt & 1]), (kt >> 1) & 1, abort_flag, err, 17)) {
        ok = false;
        break;
      }
      tc_fence_after();
      const uint32_t tS =
          tmem_base + lane_off + TM_S0 + (uint32_t)((kt & 1) * AT_BN) + (uint32_t)(half * KH);
      const int kbase = kt * AT_BN + half * KH;
      const bool full = kbase + KH <= Lk;  // no key of this half-tile is past Lk
      uint32_t sv[KH];                      // this row of S, this half of the tile
      tmem_ld32_nowait(tS, sv);
      tmem_ld32_nowait(tS + 32, sv + 32);
      tmem_ld_wait();
      if (!full) {
#pragma unroll
        for (int i = 0; i < KH; ++i)
          if (kbase + i >= Lk) sv[i] = __float_as_uint(-INFINITY);
      }
      float pm[8];
#pragma unroll
      for (int j = 0; j < 8; ++j) pm[j] = __uint_as_float(sv[j]);
#pragma unroll
      for (int i = 8; i < KH; ++i) pm[i & 7] = fmaxf(pm[i & 7], __uint_as_float(sv[i]));
      const float hmax = fmaxf(fmaxf(fmaxf(pm[0], pm[1]), fmaxf(pm[2], pm[3])),
                               fmaxf(fmaxf(pm[4], pm[5]), fmaxf(pm[6], pm[7])));
      // exchange the half-row maxima with the other warpgroup
      float* xp = xch + (kt & 1) * 2 * AT_BM;
      xp[half * AT_BM + row] = hmax;
      __syncwarp();
      if (lane == 0) mbar_arrive(su32(&xbar[kt & 1]));
      if (!warp_wait(su32(&xbar[kt & 1]), (kt >> 1) & 1, abort_flag, err, 22)) {
        ok = false;
        break;
      }
      const float mt = fmaxf(hmax, xp[(half ^ 1) * AT_BM + row]) * scale_log2;
      if (kt > 0) {
        const bool need = mt > m + 8.f;
        if (__any_sync(0xffffffffu, need)) {
          // P V of the previous tile must be complete before O is rescaled.  At
          // least P V of tile kt-2 has completed (S(kt) was issued after it),
          // and P V of tile kt needs this warp's P, so the parity names tile kt-1.
          if (!warp_wait(su32(o_done), (kt - 1) & 1, abort_flag, err, 18)) {
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
          for (int c = 0; c < HD / 64; ++c) {
            tmem_ld32(tO + c * 32, r);
#pragma unroll
            for (int i = 0; i < 32; ++i) r[i] = __float_as_uint(__uint_as_float(r[i]) * alpha);
            tmem_st32(tO + c * 32, r);
          }
          tmem_st_wait();
        }
      } else {
        m = mt;
      }
      // P = exp2(S * scale - m) for this half, two keys per TMEM column (the
      // lower key in the low 16 bits), over this half's first 32 S columns.
      float ps[8] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
      const float nm = -m;
      uint32_t pk[KH / 2];
#pragma unroll
      for (int i = 0; i < KH / 2; ++i) {
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
      if (lane == 0) mbar_arrive(su32(&p_full[kt & 1]));
    }
    // Combine the two halves' sums (one more exchange round), then O / l.
    bool fin = ok;
    if (fin) {
      float* xp = xch + (nkt & 1) * 2 * AT_BM;
      xp[half * AT_BM + row] = l;
      __syncwarp();
      if (lane == 0) mbar_arrive(su32(&xbar[nkt & 1]));
      fin = warp_wait(su32(&xbar[nkt & 1]), (nkt >> 1) & 1, abort_flag, err, 23);
      if (fin) l += xp[(half ^ 1) * AT_BM + row];
    }
    if (fin && warp_wait(su32(done), 0, abort_flag, err, 19)) {
      tc_fence_after();
      const float inv = 1.f / l;
      const int qrow = q0 + row;
      bf16* orow = O + (((int64_t)sq * Lq + qrow) * H + hq) * HD + half * (HD / 2);
      uint32_t r2[32];
#pragma unroll 1
      for (int c = 0; c < HD / 64; ++c) {
        tmem_ld32(tO + c * 32, r2);
        if (qrow < Lq) {
#pragma unroll
          for (int j = 0; j < 4; ++j) {
            uint4 v;
            v.x = pack_bf16x2(__uint_as_float(r2[8 * j]) * inv, __uint_as_float(r2[8 * j + 1]) * inv);
            v.y = pack_bf16x2(__uint_as_float(r2[8 * j + 2]) * inv, __uint_as_float(r2[8 * j + 3]) * inv);
            v.z = pack_bf16x2(__uint_as_float(r2[8 * j + 4]) * inv, __uint_as_float(r2[8 * j + 5]) * inv);
            v.w = pack_bf16x2(__uint_as_float(r2[8 * j + 6]) * inv, __uint_as_float(r2[8 * j + 7]) * inv);
            *reinterpret_cast<uint4*>(orow + c * 32 + 8 * j) = v;
          }
        }
      }
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
  dim3 grid((Lq + AT_BM - 1) / AT_BM, S_ * H);
  count_launch();
  return launch_pdl(k_attn_tc<HD>, grid, AT_THREADS, S1::SMEM, s, tq, tk, tv, (bf16*)O, H, Lq, Lk,
                    scale_log2, q_tok, k_tok, err);
}

}  // namespace

cudaError_t attention_bf16(const AttnOperand& Q, const AttnOperand& K, const AttnOperand& V,
                           void* O, int S, int H, int Lq, int Lk, int hd, cudaStream_t s) {
  if (S <= 0 || Lq <= 0) return cudaSuccess;
  if (Lk <= 0 || S * H > 65535) return cudaErrorInvalidValue;
  if ((((uintptr_t)Q.ptr) | ((uintptr_t)K.ptr) | ((uintptr_t)V.ptr) | ((uintptr_t)O)) & 15)
    return cudaErrorMisalignedAddress;
  if (hd == 128) return launch_attn_tc<128>(Q, K, V, O, S, H, Lq, Lk, s);
  if (hd == 64) return launch_attn_tc<64>(Q, K, V, O, S, H, Lq, Lk, s);
  return cudaErrorInvalidValue;
}

}  // namespace track
