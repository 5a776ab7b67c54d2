// Self- and cross-attention of the denoiser: O = softmax(Q K^T / sqrt(hd)) V per
// (sequence, head), no mask, online softmax (one pass over the keys).
//
//  * attention_bf16: the tcgen05 / TMEM flash-attention kernel of attn_tc.cu.
//  * attention_f32: true-fp32 SIMT kernel for the fp32 parity mode.
// Layouts: Q [S, H, Lq, hd], K/V [S, H, Lk, hd], O [S, Lq, H, hd] (token-major, so
// the output projection reads it as a row-major [S*Lq, H*hd] matrix).
#include <cuda_bf16.h>
#include <math.h>

#include "internal.h"

namespace track {

namespace {

typedef __nv_bfloat16 bf16;

// ---------------------------------------------------------------- fp32 SIMT
constexpr int F32_ROWS = 4;   // query rows per warp
constexpr int F32_KT = 32;    // keys per tile

template <int HD>
__global__ void __launch_bounds__(128) k_attn_f32(AttnOperand Qo, AttnOperand Ko, AttnOperand Vo,
                                                  float* __restrict__ O, int H, int Lq, int Lk,
                                                  float scale) {
  pdl_wait();
  pdl_release();
  constexpr int DV = HD / 32;
  __shared__ float sK[F32_KT][HD + 1];
  __shared__ float sV[F32_KT][HD + 1];
  __shared__ float sQ[4 * F32_ROWS][HD];
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int bh = blockIdx.y, q0 = blockIdx.x * 4 * F32_ROWS;
  const int sq = bh / H, hq = bh % H;
  const float* Qg = (const float*)Qo.ptr + sq * Qo.ss + hq * Qo.hs;
  const float* Kg = (const float*)Ko.ptr + sq * Ko.ss + hq * Ko.hs;
  const float* Vg = (const float*)Vo.ptr + sq * Vo.ss + hq * Vo.hs;
  for (int i = threadIdx.x; i < 4 * F32_ROWS * HD; i += blockDim.x) {
    const int r = i / HD, c = i % HD;
    sQ[r][c] = (q0 + r < Lq) ? Qg[(int64_t)(q0 + r) * Qo.ls + c] : 0.f;
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
      sK[r][c] = ok ? Kg[(int64_t)(k0 + r) * Ko.ls + c] : 0.f;
      sV[r][c] = ok ? Vg[(int64_t)(k0 + r) * Vo.ls + c] : 0.f;
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
#pragma unroll
  for (int i = 0; i < F32_ROWS; ++i) {
    const int row = q0 + warp * F32_ROWS + i;
    if (row >= Lq) continue;
    float* orow = O + (((int64_t)sq * Lq + row) * H + hq) * HD;
#pragma unroll
    for (int d = 0; d < DV; ++d) orow[lane + 32 * d] = o[i][d] / l[i];
  }
}

}  // namespace

cudaError_t attention_f32(const AttnOperand& Q, const AttnOperand& K, const AttnOperand& V,
                          float* O, int S, int H, int Lq, int Lk, int hd, cudaStream_t s) {
  if (S <= 0 || Lq <= 0) return cudaSuccess;
  if (Lk <= 0) return cudaErrorInvalidValue;
  dim3 grid((Lq + 4 * F32_ROWS - 1) / (4 * F32_ROWS), S * H);
  const float scale = (float)(1.0 / sqrt((double)hd));
  count_launch();
  if (hd == 128) return launch_pdl(k_attn_f32<128>, grid, 128, 0, s, Q, K, V, O, H, Lq, Lk, scale);
  if (hd == 64) return launch_pdl(k_attn_f32<64>, grid, 128, 0, s, Q, K, V, O, H, Lq, Lk, scale);
  return cudaErrorInvalidValue;
}

}  // namespace track
