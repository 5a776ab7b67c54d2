// Self- and cross-attention of the denoiser: O = softmax(Q K^T / sqrt(hd)) V per
// (sequence, head), no mask, online softmax (one pass over the keys).
//
//  * attention_bf16: flash-attention tile kernel.  64 query rows per CTA (16 per
//    warp), 64-key tiles double-buffered in shared memory with cp.async (16-byte
//    chunks, XOR-swizzled rows so ldmatrix is conflict-free), S = Q K^T and
//    O += P V on the bf16 tensor cores with fp32 accumulation, softmax in fp32
//    with exp2 and the 1/sqrt(hd) * log2(e) scale folded in.
//  * attention_f32: true-fp32 SIMT kernel for the fp32 parity mode.
// Layouts: Q [S, H, Lq, hd], K/V [S, H, Lk, hd], O [S, Lq, H, hd] (token-major, so
// the output projection reads it as a row-major [S*Lq, H*hd] matrix).
#include <cuda_bf16.h>
#include <math.h>

#include "internal.h"

namespace track {

namespace {

typedef __nv_bfloat16 bf16;

__device__ __forceinline__ uint32_t su32(const void* p) {
  return (uint32_t)__cvta_generic_to_shared(p);
}
__device__ __forceinline__ void cp_async16(uint32_t dst, const void* src, int bytes) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;" ::"r"(dst), "l"(src), "r"(bytes)
               : "memory");
}
__device__ __forceinline__ void cp_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }
template <int N>
__device__ __forceinline__ void cp_wait() {
  asm volatile("cp.async.wait_group %0;" ::"n"(N) : "memory");
}
__device__ __forceinline__ void ldsm_x4(uint32_t addr, uint32_t& r0, uint32_t& r1, uint32_t& r2,
                                        uint32_t& r3) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0, %1, %2, %3}, [%4];"
               : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
               : "r"(addr));
}
__device__ __forceinline__ void ldsm_x4_t(uint32_t addr, uint32_t& r0, uint32_t& r1, uint32_t& r2,
                                          uint32_t& r3) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0, %1, %2, %3}, [%4];"
               : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
               : "r"(addr));
}
__device__ __forceinline__ void mma16816(float (&d)[4], const uint32_t (&a)[4], uint32_t b0,
                                         uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0, %1, %2, %3}, {%4, %5, %6, %7}, "
      "{%8, %9}, {%0, %1, %2, %3};"
      : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
      : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}
__device__ __forceinline__ uint32_t pack_bf16(float lo, float hi) {
  __nv_bfloat162 t = __floats2bfloat162_rn(lo, hi);
  return *reinterpret_cast<uint32_t*>(&t);
}

constexpr int FA_BM = 64, FA_BN = 64, FA_THREADS = 128;

// Byte offset of 16-byte chunk c of row r in a tile with HD bf16 per row.
template <int HD>
__device__ __forceinline__ uint32_t swz(int r, int c) {
  return (uint32_t)(r * HD * 2 + ((c ^ (r & 7)) << 4));
}

template <int HD>
__device__ __forceinline__ void load_tile(bf16* dst, const bf16* src, int row0, int nrows, int R) {
  constexpr int CH = HD / 8;
  const uint32_t base = su32(dst);
  for (int i = threadIdx.x; i < R * CH; i += FA_THREADS) {
    const int r = i / CH, c = i % CH, gr = row0 + r;
    const bf16* gp = src + (int64_t)(gr < nrows ? gr : nrows - 1) * HD + c * 8;
    cp_async16(base + swz<HD>(r, c), gp, gr < nrows ? 16 : 0);
  }
}

template <int HD>
__global__ void __launch_bounds__(FA_THREADS, 2)
    k_attn_bf16(const bf16* __restrict__ Q, const bf16* __restrict__ K, const bf16* __restrict__ V,
                bf16* __restrict__ O, int H, int Lq, int Lk, float scale_log2) {
  constexpr int NT = FA_BN / 8;  // key n-tiles per tile
  constexpr int DT = HD / 8;     // output n-tiles
  constexpr int KS = HD / 16;    // k-steps of Q K^T
  extern __shared__ __align__(128) uint8_t fa_smem[];
  bf16* sQ = (bf16*)fa_smem;
  bf16* sK = sQ + FA_BM * HD;
  bf16* sV = sK + 2 * FA_BN * HD;

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int g = lane >> 2, t = lane & 3;
  const int bh = blockIdx.y, q0 = blockIdx.x * FA_BM;
  const bf16* Qg = Q + (int64_t)bh * Lq * HD;
  const bf16* Kg = K + (int64_t)bh * Lk * HD;
  const bf16* Vg = V + (int64_t)bh * Lk * HD;

  load_tile<HD>(sQ, Qg, q0, Lq, FA_BM);
  load_tile<HD>(sK, Kg, 0, Lk, FA_BN);
  load_tile<HD>(sV, Vg, 0, Lk, FA_BN);
  cp_commit();

  const int nkt = (Lk + FA_BN - 1) / FA_BN;
  float o[DT][4];
#pragma unroll
  for (int i = 0; i < DT; ++i) o[i][0] = o[i][1] = o[i][2] = o[i][3] = 0.f;
  float m_r[2] = {-INFINITY, -INFINITY}, l_r[2] = {0.f, 0.f};
  uint32_t qf[KS][4];
  const int mat = lane >> 3, mr = lane & 7;

  for (int kt = 0; kt < nkt; ++kt) {
    if (kt + 1 < nkt) {
      const int nb = (kt + 1) & 1;
      load_tile<HD>(sK + nb * FA_BN * HD, Kg, (kt + 1) * FA_BN, Lk, FA_BN);
      load_tile<HD>(sV + nb * FA_BN * HD, Vg, (kt + 1) * FA_BN, Lk, FA_BN);
      cp_commit();
      cp_wait<1>();
    } else {
      cp_wait<0>();
    }
    __syncthreads();
    if (kt == 0) {
#pragma unroll
      for (int kk = 0; kk < KS; ++kk) {
        const int row = warp * 16 + (mat & 1) * 8 + mr;
        ldsm_x4(su32(sQ) + swz<HD>(row, kk * 2 + (mat >> 1)), qf[kk][0], qf[kk][1], qf[kk][2],
                qf[kk][3]);
      }
    }
    const uint32_t cK = su32(sK + (kt & 1) * FA_BN * HD);
    const uint32_t cV = su32(sV + (kt & 1) * FA_BN * HD);

    float sacc[NT][4];
#pragma unroll
    for (int j = 0; j < NT; ++j) sacc[j][0] = sacc[j][1] = sacc[j][2] = sacc[j][3] = 0.f;
#pragma unroll
    for (int kk = 0; kk < KS; ++kk) {
#pragma unroll
      for (int j = 0; j < NT; j += 2) {
        uint32_t b0, b1, b2, b3;
        const int key = (j + (mat >> 1)) * 8 + mr;
        ldsm_x4(cK + swz<HD>(key, kk * 2 + (mat & 1)), b0, b1, b2, b3);
        mma16816(sacc[j], qf[kk], b0, b1);
        mma16816(sacc[j + 1], qf[kk], b2, b3);
      }
    }
    if ((kt + 1) * FA_BN > Lk) {
#pragma unroll
      for (int j = 0; j < NT; ++j)
#pragma unroll
        for (int e = 0; e < 4; ++e)
          if (kt * FA_BN + j * 8 + 2 * t + (e & 1) >= Lk) sacc[j][e] = -INFINITY;
    }
#pragma unroll
    for (int rr = 0; rr < 2; ++rr) {
      float mx = -INFINITY;
#pragma unroll
      for (int j = 0; j < NT; ++j) mx = fmaxf(mx, fmaxf(sacc[j][2 * rr], sacc[j][2 * rr + 1]));
      mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 1));
      mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 2));
      const float m_new = fmaxf(m_r[rr], mx * scale_log2);
      const float alpha = exp2f(m_r[rr] - m_new);
      m_r[rr] = m_new;
      float rs = 0.f;
#pragma unroll
      for (int j = 0; j < NT; ++j) {
        const float p0 = exp2f(fmaf(sacc[j][2 * rr], scale_log2, -m_new));
        const float p1 = exp2f(fmaf(sacc[j][2 * rr + 1], scale_log2, -m_new));
        sacc[j][2 * rr] = p0;
        sacc[j][2 * rr + 1] = p1;
        rs += p0 + p1;
      }
      l_r[rr] = l_r[rr] * alpha + rs;
#pragma unroll
      for (int n = 0; n < DT; ++n) {
        o[n][2 * rr] *= alpha;
        o[n][2 * rr + 1] *= alpha;
      }
    }
#pragma unroll
    for (int kk2 = 0; kk2 < FA_BN / 16; ++kk2) {
      uint32_t a[4];
      a[0] = pack_bf16(sacc[2 * kk2][0], sacc[2 * kk2][1]);
      a[1] = pack_bf16(sacc[2 * kk2][2], sacc[2 * kk2][3]);
      a[2] = pack_bf16(sacc[2 * kk2 + 1][0], sacc[2 * kk2 + 1][1]);
      a[3] = pack_bf16(sacc[2 * kk2 + 1][2], sacc[2 * kk2 + 1][3]);
#pragma unroll
      for (int n = 0; n < DT; n += 2) {
        uint32_t b0, b1, b2, b3;
        const int key = kk2 * 16 + (mat & 1) * 8 + mr;
        ldsm_x4_t(cV + swz<HD>(key, n + (mat >> 1)), b0, b1, b2, b3);
        mma16816(o[n], a, b0, b1);
        mma16816(o[n + 1], a, b2, b3);
      }
    }
    __syncthreads();
  }

  const int S_ = bh / H, h = bh % H;
#pragma unroll
  for (int rr = 0; rr < 2; ++rr) {
    float l = l_r[rr];
    l += __shfl_xor_sync(0xffffffffu, l, 1);
    l += __shfl_xor_sync(0xffffffffu, l, 2);
    const float inv = 1.f / l;
    const int row = q0 + warp * 16 + g + rr * 8;
    if (row < Lq) {
      bf16* orow = O + (((int64_t)S_ * Lq + row) * H + h) * HD;
#pragma unroll
      for (int n = 0; n < DT; ++n) {
        const uint32_t pk = pack_bf16(o[n][2 * rr] * inv, o[n][2 * rr + 1] * inv);
        *reinterpret_cast<uint32_t*>(orow + n * 8 + 2 * t) = pk;
      }
    }
  }
}

// ---------------------------------------------------------------- fp32 SIMT
constexpr int F32_ROWS = 4;   // query rows per warp
constexpr int F32_KT = 32;    // keys per tile

template <int HD>
__global__ void __launch_bounds__(128) k_attn_f32(const float* __restrict__ Q,
                                                  const float* __restrict__ K,
                                                  const float* __restrict__ V,
                                                  float* __restrict__ O, int H, int Lq, int Lk,
                                                  float scale) {
  constexpr int DV = HD / 32;
  __shared__ float sK[F32_KT][HD + 1];
  __shared__ float sV[F32_KT][HD + 1];
  __shared__ float sQ[4 * F32_ROWS][HD];
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int bh = blockIdx.y, q0 = blockIdx.x * 4 * F32_ROWS;
  const float* Qg = Q + (int64_t)bh * Lq * HD;
  const float* Kg = K + (int64_t)bh * Lk * HD;
  const float* Vg = V + (int64_t)bh * Lk * HD;
  for (int i = threadIdx.x; i < 4 * F32_ROWS * HD; i += blockDim.x) {
    const int r = i / HD, c = i % HD;
    sQ[r][c] = (q0 + r < Lq) ? Qg[(int64_t)(q0 + r) * HD + c] : 0.f;
  }
  float m[F32_ROWS], l[F32_ROWS], o[F32_ROWS][DV];
#pragma unroll
  for (int i = 0; i < F32_ROWS; ++i) {
    m[i] = -INFINITY;
    l[i] = 0.f;
#pragma unroll
    for (int d = 0; d < DV; ++d) o[i][d] = 0.f;
  }
  for (int k0 = 0; k0 < Lk; k0 += F32_KT) {
    __syncthreads();
    for (int i = threadIdx.x; i < F32_KT * HD; i += blockDim.x) {
      const int r = i / HD, c = i % HD;
      const bool ok = k0 + r < Lk;
      sK[r][c] = ok ? Kg[(int64_t)(k0 + r) * HD + c] : 0.f;
      sV[r][c] = ok ? Vg[(int64_t)(k0 + r) * HD + c] : 0.f;
    }
    __syncthreads();
    const bool valid = k0 + lane < Lk;
#pragma unroll
    for (int i = 0; i < F32_ROWS; ++i) {
      const int qr = warp * F32_ROWS + i;
      float s = 0.f;
#pragma unroll 8
      for (int d = 0; d < HD; ++d) s = fmaf(sQ[qr][d], sK[lane][d], s);
      s = valid ? s * scale : -INFINITY;
      float mx = s;
      for (int w = 16; w > 0; w >>= 1) mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, w));
      const float m_new = fmaxf(m[i], mx);
      const float alpha = expf(m[i] - m_new);
      const float p = valid ? expf(s - m_new) : 0.f;
      float ps = p;
      for (int w = 16; w > 0; w >>= 1) ps += __shfl_xor_sync(0xffffffffu, ps, w);
      l[i] = l[i] * alpha + ps;
      m[i] = m_new;
#pragma unroll
      for (int d = 0; d < DV; ++d) o[i][d] *= alpha;
      for (int j = 0; j < F32_KT; ++j) {
        const float pj = __shfl_sync(0xffffffffu, p, j);
#pragma unroll
        for (int d = 0; d < DV; ++d) o[i][d] = fmaf(pj, sV[j][lane + 32 * d], o[i][d]);
      }
    }
  }
  const int S_ = bh / H, h = bh % H;
#pragma unroll
  for (int i = 0; i < F32_ROWS; ++i) {
    const int row = q0 + warp * F32_ROWS + i;
    if (row >= Lq) continue;
    float* orow = O + (((int64_t)S_ * Lq + row) * H + h) * HD;
#pragma unroll
    for (int d = 0; d < DV; ++d) orow[lane + 32 * d] = o[i][d] / l[i];
  }
}

}  // namespace

cudaError_t attention_bf16(const void* Q, const void* K, const void* V, void* O, int S, int H,
                           int Lq, int Lk, int hd, cudaStream_t s) {
  if (S <= 0 || Lq <= 0) return cudaSuccess;
  if (Lk <= 0) return cudaErrorInvalidValue;
  dim3 grid((Lq + FA_BM - 1) / FA_BM, S * H);
  const float scale_log2 = (float)(1.4426950408889634 / sqrt((double)hd));
  if (hd == 128) {
    const size_t sm = (size_t)(FA_BM + 4 * FA_BN) * 128 * 2;
    cudaError_t e = cudaFuncSetAttribute(k_attn_bf16<128>,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize, (int)sm);
    if (e != cudaSuccess) return e;
    k_attn_bf16<128><<<grid, FA_THREADS, sm, s>>>((const bf16*)Q, (const bf16*)K, (const bf16*)V,
                                                   (bf16*)O, H, Lq, Lk, scale_log2);
  } else if (hd == 64) {
    const size_t sm = (size_t)(FA_BM + 4 * FA_BN) * 64 * 2;
    k_attn_bf16<64><<<grid, FA_THREADS, sm, s>>>((const bf16*)Q, (const bf16*)K, (const bf16*)V,
                                                  (bf16*)O, H, Lq, Lk, scale_log2);
  } else {
    return cudaErrorInvalidValue;
  }
  count_launch();
  return cudaGetLastError();
}

cudaError_t attention_f32(const float* Q, const float* K, const float* V, float* O, int S, int H,
                          int Lq, int Lk, int hd, cudaStream_t s) {
  if (S <= 0 || Lq <= 0) return cudaSuccess;
  if (Lk <= 0) return cudaErrorInvalidValue;
  dim3 grid((Lq + 4 * F32_ROWS - 1) / (4 * F32_ROWS), S * H);
  const float scale = (float)(1.0 / sqrt((double)hd));
  if (hd == 128) k_attn_f32<128><<<grid, 128, 0, s>>>(Q, K, V, O, H, Lq, Lk, scale);
  else if (hd == 64) k_attn_f32<64><<<grid, 128, 0, s>>>(Q, K, V, O, H, Lq, Lk, scale);
  else return cudaErrorInvalidValue;
  count_launch();
  return cudaGetLastError();
}

}  // namespace track
