// Frequency-band split of the disagreement (Sec. 4.4): the orthonormal 3-D DFT
// of D = v_S - v_L over (F, H, W), per sample and channel, with every bin's
// energy |D^(kf, kh, kw)|^2 added to one spatial band (radius of the (h, w)
// frequency in units of Nyquist against 1/3 and 2/3) and one temporal band
// (|f| frequency, same thirds); band of a bin decided in integer arithmetic.
//
// Three separable passes over shared-memory tiles, every sum in a fixed order
// (deterministic):
//   pass W  Y1[c,f,h,kw] = sum_w D[c,f,h,w] e^{-2 pi i kw w / W} / sqrt(W), with
//           per-block partial sums of v_L^2 (the denominator of Eq. 4)
//   pass H  Y2[c,f,kh,kw] = sum_h Y1[c,f,h,kw] e^{-2 pi i kh h / H} / sqrt(H)
//   pass F  Y3 = sum_f Y2[c,f,kh,kw] e^{-2 pi i kf f / F} / sqrt(F), |Y3|^2 into
//           six band partials per block
//   final   per sample, partials added in block order in fp64, then
//           sqrt(E_band) / max(||v_L||, eps).
// Twiddles come from sincospi in double, once per block.
#include <math.h>

#include "internal.h"

namespace track {

namespace {

constexpr int BD_THREADS = 256;
constexpr int BD_MAXN = 512;  // longest transformed axis supported

__device__ __forceinline__ int freq_abs(int k, int n) { return k < n - k ? k : n - k; }

__device__ __forceinline__ int spatial_band(int kh, int kw, int H, int W) {
  const int64_t a = freq_abs(kh, H), b = freq_abs(kw, W);
  const int64_t num = 4 * (a * a * W * W + b * b * H * H);
  const int64_t den = (int64_t)H * H * W * W;
  return 9 * num < den ? 0 : (9 * num < 4 * den ? 1 : 2);
}

__device__ __forceinline__ int temporal_band(int kf, int F) {
  const int a = freq_abs(kf, F);
  return 6 * a < F ? 0 : (3 * a < F ? 1 : 2);
}

// e^{-2 pi i m / n} / sqrt(n) for m = 0..n-1 into shared memory.
__device__ __forceinline__ void make_twiddles(float2* tw, int n) {
  const double scale = 1.0 / sqrt((double)n);
  for (int m = threadIdx.x; m < n; m += blockDim.x) {
    double s, c;
    sincospi(2.0 * m / n, &s, &c);
    tw[m] = make_float2((float)(c * scale), (float)(-s * scale));
  }
}

__device__ __forceinline__ float2 cmac(float2 acc, float2 a, float2 w) {
  acc.x = fmaf(a.x, w.x, fmaf(-a.y, w.y, acc.x));
  acc.y = fmaf(a.x, w.y, fmaf(a.y, w.x, acc.y));
  return acc;
}

// Block sum of v over BD_THREADS threads in a fixed order (warp shuffles, then
// warp 0 over the warp sums); the result is valid in thread 0.
__device__ __forceinline__ float block_sum(float v, float* red) {
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  __syncthreads();
  if (lane == 0) red[warp] = v;
  __syncthreads();
  float t = 0.f;
  if (warp == 0) {
    t = lane < BD_THREADS / 32 ? red[lane] : 0.f;
    for (int o = 16; o > 0; o >>= 1) t += __shfl_xor_sync(0xffffffffu, t, o);
  }
  return t;
}

// Each pass stages a tile in shared memory so every input element is read from
// global memory once, then each thread forms output bins from the tile.
constexpr int BD_COLS = 32;     // columns (innermost-axis positions) per H / F tile
constexpr int BD_ROWS_W = 16;   // rows per W tile

// grid (ceil(rows / BD_ROWS_W), B): a tile of BD_ROWS_W rows of D = v_S - v_L.
__global__ void __launch_bounds__(BD_THREADS) k_band_w(const float* __restrict__ vL,
                                                       const float* __restrict__ vS,
                                                       float2* __restrict__ Y, int64_t rows,
                                                       int W, float* __restrict__ l2part) {
  pdl_wait();
  pdl_release();
  __shared__ float2 tw[BD_MAXN];
  __shared__ float red[BD_THREADS / 32];
  extern __shared__ float dtile[];  // [BD_ROWS_W][W]
  make_twiddles(tw, W);
  const int b = blockIdx.y;
  const int64_t per = rows * W;
  const int64_t r0 = (int64_t)blockIdx.x * BD_ROWS_W;
  const int nr = (int)(rows - r0 < BD_ROWS_W ? rows - r0 : BD_ROWS_W);
  const float* dl = vL + (int64_t)b * per + r0 * W;
  const float* ds = vS + (int64_t)b * per + r0 * W;
  float l2 = 0.f;
  for (int i = threadIdx.x; i < nr * W; i += BD_THREADS) {
    const float x = dl[i];
    dtile[i] = ds[i] - x;
    l2 = fmaf(x, x, l2);
  }
  __syncthreads();
  float2* yt = Y + (int64_t)b * per + r0 * W;
  for (int o = threadIdx.x; o < nr * W; o += BD_THREADS) {
    const int r = o / W, kw = o - r * W;
    const float* d = dtile + r * W;
    float2 acc = make_float2(0.f, 0.f);
    int m = 0;  // kw * w mod W
    for (int w = 0; w < W; ++w) {
      acc.x = fmaf(d[w], tw[m].x, acc.x);
      acc.y = fmaf(d[w], tw[m].y, acc.y);
      m += kw;
      if (m >= W) m -= W;
    }
    yt[o] = acc;
  }
  const float s = block_sum(l2, red);
  if (threadIdx.x == 0) l2part[(int64_t)b * gridDim.x + blockIdx.x] = s;
}

// grid (CF * ceil(W / BD_COLS), B): columns kw0..kw0+31 of one (c, f), all H.
__global__ void __launch_bounds__(BD_THREADS) k_band_h(const float2* __restrict__ Y1,
                                                       float2* __restrict__ Y2, int CF, int H,
                                                       int W) {
  pdl_wait();
  pdl_release();
  __shared__ float2 tw[BD_MAXN];
  extern __shared__ float2 ctile[];  // [H][BD_COLS]
  make_twiddles(tw, H);
  const int ncb = (W + BD_COLS - 1) / BD_COLS;
  const int cf = blockIdx.x / ncb, kw0 = (blockIdx.x % ncb) * BD_COLS;
  const int nc = W - kw0 < BD_COLS ? W - kw0 : BD_COLS;
  const int64_t base = (int64_t)blockIdx.y * CF * H * W + (int64_t)cf * H * W + kw0;
  for (int i = threadIdx.x; i < H * BD_COLS; i += BD_THREADS) {
    const int h = i / BD_COLS, j = i % BD_COLS;
    if (j < nc) ctile[i] = Y1[base + (int64_t)h * W + j];
  }
  __syncthreads();
  for (int o = threadIdx.x; o < H * BD_COLS; o += BD_THREADS) {
    const int kh = o / BD_COLS, j = o % BD_COLS;
    if (j >= nc) continue;
    float2 acc = make_float2(0.f, 0.f);
    int m = 0;
    for (int h = 0; h < H; ++h) {
      acc = cmac(acc, ctile[h * BD_COLS + j], tw[m]);
      m += kh;
      if (m >= H) m -= H;
    }
    Y2[base + (int64_t)kh * W + j] = acc;
  }
}

// grid (C * ceil(H*W / BD_COLS), B): positions s0..s0+31 of the (h, w) plane of
// one channel, all F; six band partials per block.
__global__ void __launch_bounds__(BD_THREADS) k_band_f(const float2* __restrict__ Y2, int C,
                                                       int F, int H, int W,
                                                       float* __restrict__ bpart) {
  pdl_wait();
  pdl_release();
  __shared__ float2 tw[BD_MAXN];
  __shared__ float red[BD_THREADS / 32];
  extern __shared__ float2 ctile[];  // [F][BD_COLS]
  make_twiddles(tw, F);
  const int64_t hw = (int64_t)H * W;
  const int nsb = (int)((hw + BD_COLS - 1) / BD_COLS);
  const int c = blockIdx.x / nsb;
  const int64_t s0 = (int64_t)(blockIdx.x % nsb) * BD_COLS;
  const int nc = (int)(hw - s0 < BD_COLS ? hw - s0 : BD_COLS);
  const float2* src = Y2 + (int64_t)blockIdx.y * C * F * hw + (int64_t)c * F * hw + s0;
  for (int i = threadIdx.x; i < F * BD_COLS; i += BD_THREADS) {
    const int f = i / BD_COLS, j = i % BD_COLS;
    if (j < nc) ctile[i] = src[(int64_t)f * hw + j];
  }
  __syncthreads();
  float e[6] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
  for (int o = threadIdx.x; o < F * BD_COLS; o += BD_THREADS) {
    const int kf = o / BD_COLS, j = o % BD_COLS;
    if (j >= nc) continue;
    float2 acc = make_float2(0.f, 0.f);
    int m = 0;
    for (int f = 0; f < F; ++f) {
      acc = cmac(acc, ctile[f * BD_COLS + j], tw[m]);
      m += kf;
      if (m >= F) m -= F;
    }
    const float en = fmaf(acc.x, acc.x, acc.y * acc.y);
    const int64_t sp = s0 + j;
    const int kh = (int)(sp / W), kw = (int)(sp % W);
    const int bs = spatial_band(kh, kw, H, W), bt = 3 + temporal_band(kf, F);
#pragma unroll
    for (int q = 0; q < 6; ++q) e[q] += (q == bs || q == bt) ? en : 0.f;
  }
  float* out = bpart + ((int64_t)blockIdx.y * gridDim.x + blockIdx.x) * 6;
#pragma unroll
  for (int q = 0; q < 6; ++q) {
    const float t = block_sum(e[q], red);
    if (threadIdx.x == 0) out[q] = t;
  }
}

// One block per sample: partials in block order (fp64), then the six ratios.
__global__ void __launch_bounds__(BD_THREADS) k_band_final(const float* __restrict__ l2part,
                                                           int nl, const float* __restrict__ bpart,
                                                           int nb, float eps,
                                                           float* __restrict__ out) {
  pdl_wait();
  pdl_release();
  __shared__ double acc[7][BD_THREADS];
  const int b = blockIdx.x;
  double s[7] = {0, 0, 0, 0, 0, 0, 0};
  for (int i = threadIdx.x; i < nl; i += BD_THREADS) s[6] += (double)l2part[(int64_t)b * nl + i];
  for (int i = threadIdx.x; i < nb; i += BD_THREADS)
    for (int j = 0; j < 6; ++j) s[j] += (double)bpart[((int64_t)b * nb + i) * 6 + j];
  for (int j = 0; j < 7; ++j) acc[j][threadIdx.x] = s[j];
  __syncthreads();
  if (threadIdx.x < 7) {
    double t = 0.0;
    for (int i = 0; i < BD_THREADS; ++i) t += acc[threadIdx.x][i];
    acc[threadIdx.x][0] = t;
  }
  __syncthreads();
  if (threadIdx.x < 6) {
    const double den = fmax(sqrt(acc[6][0]), (double)eps);
    out[b * 6 + threadIdx.x] = (float)(sqrt(acc[threadIdx.x][0]) / den);
  }
}

}  // namespace

// Blocks of each pass (the W pass writes one v_L^2 partial per block, the F pass
// six band partials per block).
static int64_t blocks_w(int C, int F, int H) {
  return ((int64_t)C * F * H + BD_ROWS_W - 1) / BD_ROWS_W;
}
static int64_t blocks_f(int C, int H, int W) {
  return (int64_t)C * (((int64_t)H * W + BD_COLS - 1) / BD_COLS);
}

size_t band_scratch_floats(int B, int C, int F, int H, int W) {
  const int64_t per = (int64_t)C * F * H * W;
  return (size_t)(4 * (int64_t)B * per + (int64_t)B * (blocks_w(C, F, H) + 6 * blocks_f(C, H, W)));
}

cudaError_t band_disagreement(const float* vL, const float* vS, int B, int C, int F, int H, int W,
                              float eps, float* out, float* scratch, cudaStream_t s) {
  if (B <= 0) return cudaSuccess;
  if (F > BD_MAXN || H > BD_MAXN || W > BD_MAXN) return cudaErrorInvalidValue;
  const int64_t per = (int64_t)C * F * H * W;
  const int64_t nw = blocks_w(C, F, H), nf = blocks_f(C, H, W);
  const int64_t nh = (int64_t)C * F * ((W + BD_COLS - 1) / BD_COLS);
  if (nw > INT32_MAX || nf > INT32_MAX || nh > INT32_MAX) return cudaErrorInvalidValue;
  const size_t smem_hf = (size_t)BD_MAXN * BD_COLS * sizeof(float2);  // up to 128 KB
  cudaError_t e = cudaFuncSetAttribute(k_band_h, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       (int)smem_hf);
  if (e == cudaSuccess)
    e = cudaFuncSetAttribute(k_band_f, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem_hf);
  if (e != cudaSuccess) return e;
  float2* Y1 = reinterpret_cast<float2*>(scratch);
  float2* Y2 = Y1 + (int64_t)B * per;
  float* l2part = reinterpret_cast<float*>(Y2 + (int64_t)B * per);
  float* bpart = l2part + (int64_t)B * nw;
  e = launch_pdl(k_band_w, dim3((unsigned)nw, B), BD_THREADS,
                             (size_t)BD_ROWS_W * W * sizeof(float), s, vL, vS, Y1,
                             (int64_t)C * F * H, W, l2part);
  if (e != cudaSuccess) return e;
  e = launch_pdl(k_band_h, dim3((unsigned)nh, B), BD_THREADS, (size_t)H * BD_COLS * sizeof(float2),
                 s, (const float2*)Y1, Y2, C * F, H, W);
  if (e != cudaSuccess) return e;
  e = launch_pdl(k_band_f, dim3((unsigned)nf, B), BD_THREADS, (size_t)F * BD_COLS * sizeof(float2),
                 s, (const float2*)Y2, C, F, H, W, bpart);
  if (e != cudaSuccess) return e;
  e = launch_pdl(k_band_final, B, BD_THREADS, 0, s, (const float*)l2part, (int)nw,
                 (const float*)bpart, (int)nf, eps, out);
  if (e != cudaSuccess) return e;
  count_launch(4);
  return cudaGetLastError();
}

}  // namespace track
