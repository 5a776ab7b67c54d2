// fp32 FFMA GEMM for the fp32 parity mode: out = A[M,K] . W[N,K]^T with the
// denoiser's epilogues (bias, GELU_tanh, gated / plain residual add).  True fp32
// arithmetic (no TF32); 64x64 output tile per block, 4x4 per thread.
#include <math.h>

#include "internal.h"

namespace track {

namespace {
constexpr int TM = 64, TN = 64, TK = 16;

__device__ __forceinline__ float gelu_tanh(float u) {
  return 0.5f * u * (1.f + tanhf(0.7978845608028654f * fmaf(0.044715f * u, u * u, u)));
}

__global__ void __launch_bounds__(256) k_gemm_f32(const float* __restrict__ A,
                                                  const float* __restrict__ W, GemmArgs g) {
  pdl_wait();
  pdl_release();
  __shared__ float As[TK][TM + 4];
  __shared__ float Ws[TK][TN + 4];
  const int tid = threadIdx.x, tx = tid % 16, ty = tid / 16;
  const int row0 = blockIdx.y * TM, col0 = blockIdx.x * TN;
  float acc[4][4] = {};
  for (int k0 = 0; k0 < g.K; k0 += TK) {
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      const int idx = tid + i * 256, r = idx / TK, c = idx % TK;
      const int gr = row0 + r, gn = col0 + r, gk = k0 + c;
      As[c][r] = (gr < g.M && gk < g.K) ? A[(int64_t)gr * g.K + gk] : 0.f;
      Ws[c][r] = (gn < g.N && gk < g.K) ? W[(int64_t)gn * g.K + gk] : 0.f;
    }
    __syncthreads();
#pragma unroll
    for (int kk = 0; kk < TK; ++kk) {
      float a[4], b[4];
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        a[i] = As[kk][ty * 4 + i];
        b[i] = Ws[kk][tx * 4 + i];
      }
#pragma unroll
      for (int i = 0; i < 4; ++i)
#pragma unroll
        for (int j = 0; j < 4; ++j) acc[i][j] = fmaf(a[i], b[j], acc[i][j]);
    }
    __syncthreads();
  }
  float* out = (float*)g.out;
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const int r = row0 + ty * 4 + i;
    if (r >= g.M) continue;
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const int c = col0 + tx * 4 + j;
      if (c >= g.N) continue;
      float v = acc[i][j] + (g.bias ? g.bias[c] : 0.f);
      float* o = out + (int64_t)r * g.ldo + c;
      if (g.epi == EPI_STORE) *o = v;
      else if (g.epi == EPI_GELU) *o = gelu_tanh(v);
      else if (g.epi == EPI_RESID_GATE) *o = fmaf(g.gate[c], v, *o);
      else *o = *o + v;
    }
  }
}
}  // namespace

cudaError_t gemm_f32(const float* A, const float* W, const GemmArgs& g, cudaStream_t s) {
  if (g.M <= 0 || g.N <= 0) return cudaSuccess;
  dim3 grid((g.N + TN - 1) / TN, (g.M + TM - 1) / TM);
  if (grid.y > 65535) return cudaErrorInvalidConfiguration;
  count_launch();
  return launch_pdl(k_gemm_f32, grid, 256, 0, s, A, W, g);
}

}  // namespace track
