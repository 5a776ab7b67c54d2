// bf16 GEMM on the sm_103a tensor cores: out = A[M,K] . W[N,K]^T (+ epilogue).
//
// Persistent, warp-specialised kernel, one CTA per SM:
//   warp 0      TMA producer: 128x64 A tile and BNx64 W tile per stage into a
//               STAGES-deep shared-memory ring (128-byte swizzle, zero fill past
//               the matrix edges), completion counted on an mbarrier.
//   warp 1      allocates 2*BN TMEM columns (two fp32 128xBN accumulators) and
//               issues tcgen05.mma (kind::f16, M=128, N=BN, K=16) from one
//               thread; tcgen05.commit frees a stage / publishes an accumulator.
//   warps 2-5   epilogue: tcgen05.ld 32 columns at a time from their TMEM lane
//               quarter, add bias, apply GELU / gate / residual, store to HBM,
//               then release the accumulator so the next tile's MMAs overlap
//               this tile's epilogue.
// Every mbarrier wait is bounded: on expiry the CTA raises an abort flag,
// records an error code in the device error word, skips its remaining work,
// frees its TMEM and exits.
#include <cuda.h>
#include <cuda_bf16.h>
#include <math.h>

#include <mutex>

#include "internal.h"
#include "tc_common.cuh"

namespace track {

namespace {

using namespace tc;
typedef __nv_bfloat16 bf16;
constexpr int BM = 128, BK = 64;

__device__ __forceinline__ float gelu_tanh(float u) {
  return 0.5f * u * (1.f + tanhf(0.7978845608028654f * fmaf(0.044715f * u, u * u, u)));
}

// Writes this thread's 128-byte row `row` (8 chunks of 16 bytes) into a staging
// box in the 128-byte-swizzled layout TMA expects: chunk j at j ^ (row % 8).
__device__ __forceinline__ void stage_row(uint8_t* box, int row, const uint4 (&chunk)[8]) {
  uint8_t* base = box + row * 128;
#pragma unroll
  for (int j = 0; j < 8; ++j)
    *reinterpret_cast<uint4*>(base + ((j ^ (row & 7)) << 4)) = chunk[j];
}

__device__ __forceinline__ uint32_t pack2(float a, float b) {
  __nv_bfloat162 t = __floats2bfloat162_rn(a, b);
  return *reinterpret_cast<uint32_t*>(&t);
}

template <int BN, int STAGES>
struct TcShape {
  static constexpr uint32_t A_BYTES = BM * BK * 2;
  static constexpr uint32_t B_BYTES = BN * BK * 2;
  // two accumulators of BN columns; TMEM is allocated in powers of two columns
  static constexpr uint32_t TMEM_COLS = 2 * BN <= 256 ? 256 : 512;
  static constexpr uint32_t STG_BYTES = 4 * 2 * 4096;  // two 32x128-byte boxes per epilogue warp
  static constexpr size_t SMEM = 1024 + (size_t)STAGES * (A_BYTES + B_BYTES) + STG_BYTES + 256;
};

template <int BN, int STAGES>
__global__ void __launch_bounds__(192, 1)
    k_gemm_tc(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB,
              const __grid_constant__ CUtensorMap tmC, const GemmArgs g) {
  using S = TcShape<BN, STAGES>;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = (uint8_t*)(((uintptr_t)smem_raw + 1023) & ~(uintptr_t)1023);
  uint8_t* sA = smem;
  uint8_t* sB = smem + STAGES * S::A_BYTES;
  uint8_t* stg_all = sB + STAGES * S::B_BYTES;  // 1024-byte aligned
  uint64_t* bars = (uint64_t*)(stg_all + S::STG_BYTES);
  uint64_t* full = bars;
  uint64_t* empty = bars + STAGES;
  uint64_t* accf = bars + 2 * STAGES;
  uint64_t* acce = accf + 2;
  uint64_t* done = acce + 2;
  uint32_t* tmem_slot = (uint32_t*)(done + 1);
  volatile int* abort_flag = (volatile int*)(tmem_slot + 1);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int m_tiles = (g.M + BM - 1) / BM, n_tiles = (g.N + BN - 1) / BN;
  const int num_tiles = m_tiles * n_tiles;
  const int nk = g.K / BK;

  if (threadIdx.x == 0) {
    for (int i = 0; i < STAGES; ++i) {
      mbar_init(su32(&full[i]), 1);
      mbar_init(su32(&empty[i]), 1);
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(su32(&accf[i]), 1);
      mbar_init(su32(&acce[i]), 4);
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
  // The prologue above overlaps the previous kernel; inputs and outputs are touched only now.
  pdl_wait();
  pdl_release();

  if (warp == 0) {
    if (lane == 0) {
      asm volatile("prefetch.tensormap [%0];" ::"l"((uint64_t)&tmA) : "memory");
      asm volatile("prefetch.tensormap [%0];" ::"l"((uint64_t)&tmB) : "memory");
      int stage = 0;
      uint32_t phase = 0;
      uint32_t armed[STAGES];
#pragma unroll
      for (int i = 0; i < STAGES; ++i) armed[i] = 0;
      for (int tile = blockIdx.x; tile < num_tiles; tile += gridDim.x) {
        const int mt = tile % m_tiles, nt = tile / m_tiles;
        bool ok = true;
        for (int kb = 0; kb < nk; ++kb) {
          if (!mbar_wait(su32(&empty[stage]), phase ^ 1, abort_flag, g.err, 1)) {
            ok = false;
            break;
          }
          const uint32_t fb = su32(&full[stage]);
          mbar_expect_tx(fb, S::A_BYTES + S::B_BYTES);
          tma_load_2d(su32(sA + stage * S::A_BYTES), &tmA, kb * BK, mt * BM, fb);
          tma_load_2d(su32(sB + stage * S::B_BYTES), &tmB, kb * BK, nt * BN, fb);
          ++armed[stage];
          if (++stage == STAGES) {
            stage = 0;
            phase ^= 1;
          }
        }
        if (!ok) break;
      }
      // Every copy this thread issued has landed before the CTA may exit.
#pragma unroll
      for (int i = 0; i < STAGES; ++i)
        if (armed[i] != 0) mbar_drain(su32(&full[i]), (armed[i] - 1) & 1, g.err, 5);
    }
  } else if (warp == 1) {
    if (lane == 0) {
      constexpr uint32_t idesc = idesc_bf16(BM, BN);
      int stage = 0, acc = 0;
      uint32_t phase = 0, acc_phase = 0;
      for (int tile = blockIdx.x; tile < num_tiles; tile += gridDim.x) {
        if (!mbar_wait(su32(&acce[acc]), acc_phase ^ 1, abort_flag, g.err, 2)) break;
        tc_fence_after();
        const uint32_t d_tmem = tmem_base + (uint32_t)(acc * BN);
        bool ok = true;
        for (int kb = 0; kb < nk; ++kb) {
          if (!mbar_wait(su32(&full[stage]), phase, abort_flag, g.err, 3)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t a0 = su32(sA + stage * S::A_BYTES);
          const uint32_t b0 = su32(sB + stage * S::B_BYTES);
#pragma unroll
          for (int k = 0; k < BK / 16; ++k)
            mma_bf16(d_tmem, sdesc_sw128(a0 + k * 32), sdesc_sw128(b0 + k * 32), idesc,
                     (kb | k) != 0 ? 1u : 0u);
          mma_commit(su32(&empty[stage]));
          if (++stage == STAGES) {
            stage = 0;
            phase ^= 1;
          }
        }
        if (!ok) break;
        mma_commit(su32(&accf[acc]));
        if (++acc == 2) {
          acc = 0;
          acc_phase ^= 1;
        }
      }
      // Every MMA this thread issued has completed before TMEM is freed.
      mma_commit(su32(done));
      mbar_drain(su32(done), 0, g.err, 6);
    }
  } else {
    const int quarter = warp & 3;  // TMEM lanes 32*quarter .. 32*quarter+31
    uint8_t* stg = stg_all + (warp - 2) * 2 * 4096;
    const bool bf16_out = g.epi == EPI_STORE || g.epi == EPI_GELU;
    const int cw = bf16_out ? 64 : 32;  // columns per staged box (128-byte rows)
    int sb = 0, acc = 0;
    uint32_t acc_phase = 0;
    for (int tile = blockIdx.x; tile < num_tiles; tile += gridDim.x) {
      const int mt = tile % m_tiles, nt = tile / m_tiles;
      int ok = 1;
      if (lane == 0) ok = mbar_wait(su32(&accf[acc]), acc_phase, abort_flag, g.err, 4) ? 1 : 0;
      ok = __shfl_sync(0xffffffffu, ok, 0);  // the whole warp takes the same branch
      if (!ok) break;
      tc_fence_after();
      const int row_base = mt * BM + quarter * 32;
      const uint32_t tbase = tmem_base + ((uint32_t)(quarter * 32) << 16) + (uint32_t)(acc * BN);
#pragma unroll 1
      for (int c = 0; c < BN; c += cw) {
        const int col0 = nt * BN + c;
        if (row_base >= g.M || col0 >= g.N) continue;  // uniform across the warp
        uint4 chunk[8];
        if (bf16_out) {
          uint32_t r0[32], r1[32];
          tmem_ld32(tbase + (uint32_t)c, r0);
          tmem_ld32(tbase + (uint32_t)(c + 32), r1);
          const float4* b4 = reinterpret_cast<const float4*>(g.bias + col0);
          const bool gelu = g.epi == EPI_GELU;
#pragma unroll
          for (int j = 0; j < 8; ++j) {
            float v[8];
#pragma unroll
            for (int e = 0; e < 8; ++e) {
              const int i = 8 * j + e;
              v[e] = __uint_as_float(i < 32 ? r0[i] : r1[i - 32]);
            }
            if (g.bias != nullptr && (j < 4 || col0 + 64 <= g.N)) {  // columns >= N are clipped
              const float4 ba = b4[2 * j], bb = b4[2 * j + 1];
              v[0] += ba.x; v[1] += ba.y; v[2] += ba.z; v[3] += ba.w;
              v[4] += bb.x; v[5] += bb.y; v[6] += bb.z; v[7] += bb.w;
            }
            if (gelu) {
#pragma unroll
              for (int e = 0; e < 8; ++e) v[e] = gelu_tanh(v[e]);
            }
            chunk[j] = make_uint4(pack2(v[0], v[1]), pack2(v[2], v[3]), pack2(v[4], v[5]),
                                  pack2(v[6], v[7]));
          }
        } else {
          uint32_t r0[32];
          tmem_ld32(tbase + (uint32_t)c, r0);
          const float4* b4 = reinterpret_cast<const float4*>(g.bias + col0);
          const float4* g4 = reinterpret_cast<const float4*>(g.gate + col0);
          const bool gated = g.epi == EPI_RESID_GATE;
#pragma unroll
          for (int j = 0; j < 8; ++j) {
            float4 v = make_float4(__uint_as_float(r0[4 * j]), __uint_as_float(r0[4 * j + 1]),
                                   __uint_as_float(r0[4 * j + 2]), __uint_as_float(r0[4 * j + 3]));
            if (g.bias != nullptr) {
              const float4 b = b4[j];
              v.x += b.x; v.y += b.y; v.z += b.z; v.w += b.w;
            }
            if (gated) {
              const float4 gg = g4[j];
              v.x *= gg.x; v.y *= gg.y; v.z *= gg.z; v.w *= gg.w;
            }
            chunk[j] = make_uint4(__float_as_uint(v.x), __float_as_uint(v.y),
                                  __float_as_uint(v.z), __float_as_uint(v.w));
          }
        }
        // The box written two stores ago must have been read out by its TMA.
        if (lane == 0) bulk_wait_read_1();
        __syncwarp();
        uint8_t* box = stg + sb * 4096;
        stage_row(box, lane, chunk);
        fence_async_shared();
        __syncwarp();
        if (lane == 0) {
          if (bf16_out) tma_store_2d(&tmC, col0, row_base, su32(box));
          else tma_reduce_add_2d(&tmC, col0, row_base, su32(box));
          bulk_commit();
        }
        sb ^= 1;
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(su32(&acce[acc]));
      if (++acc == 2) {
        acc = 0;
        acc_phase ^= 1;
      }
    }
    if (lane == 0) bulk_wait_all();  // this warp's stores have completed
    __syncwarp();
  }

  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  if (warp == 1) {
    __syncwarp();
    tmem_dealloc(tmem_base, S::TMEM_COLS);
  }
}

// 2-D tensor map of a row-major [rows, cols] matrix with leading dimension ld
// (elements), box [box_rows, box_cols], 128-byte swizzle, zero fill out of bounds.
bool make_tmap(CUtensorMap* tm, CUtensorMapDataType dt, size_t esize, const void* ptr,
               uint64_t rows, uint64_t cols, uint64_t ld, uint32_t box_rows, uint32_t box_cols) {
  EncodeTiledFn enc = encode_tiled_fn();
  if (enc == nullptr) return false;
  cuuint64_t dims[2] = {cols, rows};
  cuuint64_t strides[1] = {ld * esize};
  cuuint32_t box[2] = {box_cols, box_rows};
  cuuint32_t estr[2] = {1, 1};
  return enc(tm, dt, 2, const_cast<void*>(ptr), dims, strides, box, estr,
             CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
             CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

template <int BN, int STAGES>
cudaError_t launch_tc(const void* A, const void* W, const GemmArgs& g, cudaStream_t s) {
  using S = TcShape<BN, STAGES>;
  static_assert(S::SMEM <= 232448, "shared memory budget");
  CUtensorMap ta, tb, tc;
  const CUtensorMapDataType BF = CU_TENSOR_MAP_DATA_TYPE_BFLOAT16;
  if (!make_tmap(&ta, BF, 2, A, (uint64_t)g.M, (uint64_t)g.K, (uint64_t)g.K, BM, BK))
    return cudaErrorInvalidValue;
  if (!make_tmap(&tb, BF, 2, W, (uint64_t)g.N, (uint64_t)g.K, (uint64_t)g.K, BN, BK))
    return cudaErrorInvalidValue;
  const bool bf16_out = g.epi == EPI_STORE || g.epi == EPI_GELU;
  if (bf16_out ? !make_tmap(&tc, BF, 2, g.out, (uint64_t)g.M, (uint64_t)g.N, (uint64_t)g.ldo, 32, 64)
               : !make_tmap(&tc, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 4, g.out, (uint64_t)g.M,
                            (uint64_t)g.N, (uint64_t)g.ldo, 32, 32))
    return cudaErrorInvalidValue;
  cudaError_t e = cudaFuncSetAttribute(k_gemm_tc<BN, STAGES>,
                                       cudaFuncAttributeMaxDynamicSharedMemorySize, (int)S::SMEM);
  if (e != cudaSuccess) return e;
  const int tiles = ((g.M + BM - 1) / BM) * ((g.N + BN - 1) / BN);
  const int grid = tiles < num_sms() ? tiles : num_sms();
  count_launch();
  return launch_pdl(k_gemm_tc<BN, STAGES>, grid, 192, S::SMEM, s, ta, tb, tc, g);
}

}  // namespace

EncodeTiledFn encode_tiled_fn() {
  static EncodeTiledFn fn = []() -> EncodeTiledFn {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault,
                                         &q) != cudaSuccess ||
        q != cudaDriverEntryPointSuccess)
      return nullptr;
    return (EncodeTiledFn)p;
  }();
  return fn;
}

cudaError_t gemm_bf16_tc(const void* A, const void* W, const GemmArgs& g, cudaStream_t s) {
  if (g.M <= 0 || g.N <= 0) return cudaSuccess;
  if (g.K <= 0 || g.K % BK != 0 || g.N % 32 != 0 || g.ldo % 8 != 0) return cudaErrorInvalidValue;
  if ((((uintptr_t)A) | ((uintptr_t)W) | ((uintptr_t)g.out)) & 15) return cudaErrorMisalignedAddress;
  if (g.bias != nullptr && (((uintptr_t)g.bias) & 15)) return cudaErrorMisalignedAddress;
  if (g.epi == EPI_RESID_GATE && (g.gate == nullptr || (((uintptr_t)g.gate) & 15)))
    return cudaErrorInvalidValue;
  // Tile width by a makespan model: every CTA of a wave runs concurrently, so a
  // launch costs about rounds x (BN + per-tile overhead).  The overhead (150
  // columns' worth) is fitted to measured tile times: a 192-wide tile takes about
  // 0.85x the time of a 256-wide one.  Ties go to the wider tile.
  const int m_tiles = (g.M + BM - 1) / BM, sms = num_sms();
  const bool fp32_out = g.epi == EPI_RESID || g.epi == EPI_RESID_GATE;  // 32-column epilogue chunks
  int best_bn = 256;
  long best_cost = -1;
  for (int bn : {256, 192, 160, 128}) {
    if (bn == 160 && !fp32_out) continue;  // bf16 epilogue chunks are 64 columns wide
    const long tiles = (long)m_tiles * ((g.N + bn - 1) / bn);
    const long cost = ((tiles + sms - 1) / sms) * (bn + 150);
    if (best_cost < 0 || cost < best_cost) {
      best_cost = cost;
      best_bn = bn;
    }
  }
  if (best_bn == 256) return launch_tc<256, 4>(A, W, g, s);
  if (best_bn == 192) return launch_tc<192, 4>(A, W, g, s);
  if (best_bn == 160) return launch_tc<160, 5>(A, W, g, s);
  return launch_tc<128, 6>(A, W, g, s);
}

}  // namespace track
