// bf16 GEMM on the sm_103a tensor cores: out = A[M,K] . W[N,K]^T (+ epilogue).
//
// Persistent, warp-specialised kernel, one CTA per SM.  A CTA follows one of
// two schedules:
//   data-parallel  CTA w takes output tiles w, w + G, ... (whole K loop);
//   stream-K       tiles of all full waves but the last are taken whole and
//                  round-robin; the remaining tiles' k-blocks form one
//                  sequence of U units and CTA w takes the contiguous share
//                  [w U / G, (w+1) U / G), so every CTA does the same number
//                  of k-blocks whatever the tile count (sharing out every tile
//                  this way would scatter the tiles in flight over the whole
//                  output and defeat L2 reuse of A and W at large sizes).  A
//                  tile split across CTAs is finished by whichever
//                  ends its part last: the others write their fp32 partial
//                  sums to a workspace slot and count in on a per-(tile, warp)
//                  counter; the last one adds the parts in k order (a fixed
//                  order, so the result does not depend on timing), applies
//                  the epilogue and resets the counter for the next launch.
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

#include <atomic>
#include <map>
#include <mutex>
#include <utility>

#include "internal.h"
#include "tc_common.cuh"

namespace track {

namespace {

using namespace tc;
typedef __nv_bfloat16 bf16;
constexpr int BM = 128, BK = 64;

// GELU, tanh form: 0.5 u (1 + tanh z) with z = sqrt(2/pi) (u + 0.044715 u^3),
// evaluated as u / (1 + e^(-2z)) (the same function; no cancellation for
// negative u) with the fast exp and divide intrinsics (about 1e-6 relative).
__device__ __forceinline__ float gelu_tanh(float u) {
  const float z = 0.7978845608028654f * fmaf(0.044715f * u, u * u, u);
  return __fdividef(u, 1.f + __expf(-2.f * z));
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

// Stream-K state: counters [4 * CTA tiles] (zero between launches) and 2 * grid
// partial-sum slots of 128 x BN floats.  cnt == nullptr selects data-parallel.
struct SkArgs {
  int* cnt;
  float* ws;
  int64_t units;  // k-blocks of the stream-K tiles (tiles dp_tiles .. end)
  int dp_tiles;   // leading tiles taken whole, round-robin
};

constexpr int SK_MAX_PARTS = 4;     // the host only picks stream-K when no tile spans more workers
// Makespan-model cost of the stream-K fix-up (publishing a partial tile, the
// counter round trips and the final combine: about 8 us), in the model's units
// of one 64-deep k-block of a 256-wide tile = 406 (about 0.33 us).
constexpr double SK_FIXUP = 10000.0;

// Work tile -> (row unit, column tile).  Tiles are numbered in groups of
// `group` row units: inside a group the row unit varies fastest, then the
// column tile.  The ~152 tiles in flight at a time then span `group` row units
// and 152/group column tiles, whose A and W blocks stay in L2 while they are
// reused, instead of one column of up to all row units, which streams all of A
// from DRAM once per column tile when A is larger than L2.  With at most
// `group` row units (3510 tokens: 28) this is the plain column order.
// Measured at 65520 rows (the 14B shapes with CFG): groups of 32 made every
// projection 13-25 % faster than column order (qkv 1813, out_proj 1542,
// cross_q 1623, ffn_up 1610, ffn_down 1534 TFLOP/s), and were the best or
// within 1 % of the best of 4, 8, 16, 32 and 64.
constexpr int RASTER_DEFAULT = 32;

__device__ __forceinline__ void tile_coords(int tile, int m_units, int n_tiles, int group, int& mu,
                                            int& nt) {
  if (group > m_units) group = m_units;  // per_group <= the tile count: no overflow
  const int per_group = group * n_tiles;
  const int g = tile / per_group;
  const int first = g * group;
  const int rows = m_units - first < group ? m_units - first : group;
  const int local = tile - g * per_group;
  mu = first + local % rows;
  nt = local / rows;
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
              const __grid_constant__ CUtensorMap tmC, const GemmArgs g, const SkArgs sk) {
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
  const int worker = blockIdx.x, workers = gridDim.x;
  const int n_tiles = (g.N + BN - 1) / BN;
  const int m_units = (g.M + BM - 1) / BM;  // row tiles
  const int num_tiles = m_units * n_tiles;
  const int nk = g.K / BK;
  const bool use_sk = sk.cnt != nullptr;

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
  // The prologue above overlaps the previous kernel; inputs and outputs are touched only
  // after the grid dependency wait.  For model weights (g.w_static) the producer thread
  // first requests the W tiles of its first stages: no kernel writes them.
  const bool producer = warp == 0 && lane == 0;
  if (!producer) {
    pdl_wait();
    pdl_release();
  }

  if (warp == 0) {
    if (lane == 0) {
      asm volatile("prefetch.tensormap [%0];" ::"l"((uint64_t)&tmA) : "memory");
      asm volatile("prefetch.tensormap [%0];" ::"l"((uint64_t)&tmB) : "memory");
      int stage = 0;
      uint32_t phase = 0;
      uint32_t armed[STAGES];
#pragma unroll
      for (int i = 0; i < STAGES; ++i) armed[i] = 0;
      SegIter it(use_sk, sk.units, num_tiles, nk, worker, workers, sk.dp_tiles);
      int pre = 0;  // k-blocks of the first segment whose W tile is already requested
      if (g.w_static) {
        SegIter first = it;
        int t0, a0, a1;
        if (first.next(t0, a0, a1)) {
          int mu0, nt0;
          tile_coords(t0, m_units, n_tiles, g.raster, mu0, nt0);
          pre = a1 - a0 < STAGES ? a1 - a0 : STAGES;
          for (int i = 0; i < pre; ++i) {  // fresh stages: no empty wait
            const uint32_t fb = su32(&full[i]);
            mbar_expect_tx(fb, S::A_BYTES + S::B_BYTES);
            tma_load_2d(su32(sB + i * S::B_BYTES), &tmB, (a0 + i) * BK, nt0 * BN, fb);
          }
        }
      }
      pdl_wait();
      pdl_release();
      int tile, kb0, kb1;
      while (it.next(tile, kb0, kb1)) {
        int mu, nt;
        tile_coords(tile, m_units, n_tiles, g.raster, mu, nt);
        const int mt = mu;
        bool ok = true;
        for (int kb = kb0; kb < kb1; ++kb) {
          const uint32_t fb = su32(&full[stage]);
          if (pre > 0) {  // W of this stage requested before the dependency wait
            --pre;
            tma_load_2d(su32(sA + stage * S::A_BYTES), &tmA, kb * BK, mt * BM, fb);
            ++armed[stage];
            if (++stage == STAGES) {
              stage = 0;
              phase ^= 1;
            }
            continue;
          }
          if (!mbar_wait(su32(&empty[stage]), phase ^ 1, abort_flag, g.err, 1)) {
            ok = false;
            break;
          }
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
      // Every copy into this CTA has landed before the CTA may exit.
#pragma unroll
      for (int i = 0; i < STAGES; ++i) {
        if (armed[i] == 0) continue;
        mbar_drain(su32(&full[i]), (armed[i] - 1) & 1, g.err, 5);
      }
    }
  } else if (warp == 1) {
    if (lane == 0) {
      constexpr uint32_t idesc = idesc_bf16(BM, BN);
      int stage = 0, acc = 0;
      uint32_t phase = 0, acc_phase = 0;
      SegIter it(use_sk, sk.units, num_tiles, nk, worker, workers, sk.dp_tiles);
      int tile, kb0, kb1;
      while (it.next(tile, kb0, kb1)) {
        if (!mbar_wait(su32(&acce[acc]), acc_phase ^ 1, abort_flag, g.err, 2)) break;
        tc_fence_after();
        const uint32_t d_tmem = tmem_base + (uint32_t)(acc * BN);
        bool ok = true;
        for (int kb = kb0; kb < kb1; ++kb) {
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
                     (kb > kb0 || k != 0) ? 1u : 0u);
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
    int sb = 0, acc = 0;
    uint32_t acc_phase = 0;
    const int64_t U = sk.units;
    constexpr int SLOT = BM * BN;  // floats per partial-sum slot
    SegIter it(use_sk, U, num_tiles, nk, worker, workers, sk.dp_tiles);
    int tile, kb0, kb1;
    while (it.next(tile, kb0, kb1)) {
      int mu, nt;
      tile_coords(tile, m_units, n_tiles, g.raster, mu, nt);
      const int mt = mu;
      const bool final_seg = it.done();
      // Bias and gate of this tile's columns are pulled into L1 while the MMAs run
      // (lane l: columns 8l..8l+7); the column loop below reads them with
      // warp-uniform loads, which L1 broadcasts.
      {
        const int cb = nt * BN + 8 * lane;
        if (8 * lane < BN && cb < g.N) {
          if (g.bias != nullptr) asm volatile("prefetch.global.L1 [%0];" ::"l"(g.bias + cb));
          if (g.epi == EPI_RESID_GATE) asm volatile("prefetch.global.L1 [%0];" ::"l"(g.gate + cb));
        }
      }
      int ok = 1;
      if (lane == 0) ok = mbar_wait(su32(&accf[acc]), acc_phase, abort_flag, g.err, 4) ? 1 : 0;
      ok = __shfl_sync(0xffffffffu, ok, 0);  // the whole warp takes the same branch
      if (!ok) break;
      tc_fence_after();
      const int row_base = mt * BM + quarter * 32;
      const uint32_t tbase = tmem_base + ((uint32_t)(quarter * 32) << 16) + (uint32_t)(acc * BN);
      // Stream-K parts of this work tile: workers w_first .. w_first + nparts - 1 in k order.
      int nparts = 1, part = 0, w_first = 0;
      bool finish = true, staged = false;
      // Partial-sum slot of part i: 2w for worker w's first
      // segment, 2w+1 for its last.
      auto slot_of = [&](int i) -> float4* {
        const int wi = w_first + i;
        const int first_tile = sk.dp_tiles + (int)(((int64_t)wi * U / workers) / nk);
        const int s = 2 * wi + (first_tile == tile ? 0 : 1);
        return reinterpret_cast<float4*>(sk.ws + (size_t)s * SLOT);
      };
      const int rowq = quarter * 32 + lane;  // this thread's row within the tile
      if (kb0 != 0 || kb1 != nk) {
        const int64_t tu = (int64_t)(tile - sk.dp_tiles) * nk;  // the tile's first unit
        w_first = sk_worker_of(tu, U, workers);
        nparts = sk_worker_of(tu + nk - 1, U, workers) - w_first + 1;
        part = worker - w_first;
        if (nparts > SK_MAX_PARTS) {  // excluded by the host's choice of schedule
          if (lane == 0) {
            *abort_flag = 1;
            atomicExch(g.err, 7);
          }
          break;
        }
        int* cnt = sk.cnt + 4 * tile + quarter;
        int last = 0;
        if (lane == 0) last = ld_acquire(cnt) == nparts - 1 ? 1 : 0;
        last = __shfl_sync(0xffffffffu, last, 0);
        if (!last) {
          // Publish this part: rows of this warp, 32-column chunks, chunk-major so
          // that each store instruction of the warp covers 512 contiguous bytes.
          float4* mine = slot_of(part);
          if (row_base < g.M) {
#pragma unroll 1
            for (int c = 0; c < BN; c += 32) {
              if (nt * BN + c >= g.N) break;
              uint32_t r[32];
              tmem_ld32(tbase + (uint32_t)c, r);
#pragma unroll
              for (int j = 0; j < 8; ++j)
                mine[((c >> 5) * 8 + j) * BM + rowq] =
                    make_float4(__uint_as_float(r[4 * j]), __uint_as_float(r[4 * j + 1]),
                                __uint_as_float(r[4 * j + 2]), __uint_as_float(r[4 * j + 3]));
            }
          }
          __threadfence();
          __syncwarp();
          if (lane == 0) last = atomicAdd(cnt, 1) == nparts - 1 ? 1 : 0;
          last = __shfl_sync(0xffffffffu, last, 0);
        }
        finish = last != 0;
        if (finish) {
          __threadfence();  // the other parts' stores are visible to this warp's loads
          if (lane == 0) *cnt = 0;  // every part has counted in: reset for the next launch
          // After the worker's last segment the operand stages are idle (every load
          // was consumed by an MMA that has completed), so the one other part is
          // copied into this warp's 32 KB of them in a single asynchronous batch.
          if (final_seg && nparts == 2 && row_base < g.M) {
            const float4* src = slot_of(1 - part) + rowq;
            const uint32_t dst = su32(smem) + (uint32_t)(warp - 2) * 32768u + lane * 16u;
            fence_async_shared();  // after the tensor core's reads of these stages
#pragma unroll 1
            for (int c = 0; c < BN; c += 32) {
              if (nt * BN + c >= g.N) break;
#pragma unroll
              for (int j = 0; j < 8; ++j)
                cp_async16(dst + (uint32_t)(((c >> 5) * 8 + j) * 512), src + ((c >> 5) * 8 + j) * BM);
            }
            cp_async_wait_all();
            staged = true;
          }
        }
      }
      // Adds the other parts' columns c..c+31 of this thread's row to its own (in r),
      // in k order: p_0 + p_1 + ... with this CTA's part at index `part` (fp32
      // addition is commutative, so t + own and own + t are the same bits).  A
      // part's eight loads are issued together: one memory latency per part.
      auto combine32 = [&](int c, uint32_t (&r)[32]) {
        float4 t[8];
#pragma unroll 1
        for (int i = 0; i < nparts; ++i) {
          if (i == part) {
            if (i > 0) {
#pragma unroll
              for (int j = 0; j < 8; ++j) {
                r[4 * j] = __float_as_uint(t[j].x + __uint_as_float(r[4 * j]));
                r[4 * j + 1] = __float_as_uint(t[j].y + __uint_as_float(r[4 * j + 1]));
                r[4 * j + 2] = __float_as_uint(t[j].z + __uint_as_float(r[4 * j + 2]));
                r[4 * j + 3] = __float_as_uint(t[j].w + __uint_as_float(r[4 * j + 3]));
              }
            }
            continue;
          }
          float4 x[8];
          if (staged) {
            const float4* src = reinterpret_cast<const float4*>(smem + (warp - 2) * 32768) +
                                (c >> 5) * 8 * 32 + lane;
#pragma unroll
            for (int j = 0; j < 8; ++j) x[j] = src[j * 32];
          } else {
            const float4* src = slot_of(i) + (c >> 5) * 8 * BM + rowq;
#pragma unroll
            for (int j = 0; j < 8; ++j) x[j] = __ldcg(src + j * BM);
          }
#pragma unroll
          for (int j = 0; j < 8; ++j) {
            if (i < part) {  // running sum of the parts before this CTA's
              if (i == 0) {
                t[j] = x[j];
              } else {
                t[j].x += x[j].x; t[j].y += x[j].y; t[j].z += x[j].z; t[j].w += x[j].w;
              }
            } else {  // parts after this CTA's: add onto the running total in r
              r[4 * j] = __float_as_uint(__uint_as_float(r[4 * j]) + x[j].x);
              r[4 * j + 1] = __float_as_uint(__uint_as_float(r[4 * j + 1]) + x[j].y);
              r[4 * j + 2] = __float_as_uint(__uint_as_float(r[4 * j + 2]) + x[j].z);
              r[4 * j + 3] = __float_as_uint(__uint_as_float(r[4 * j + 3]) + x[j].w);
            }
          }
        }
      };
      // Stages 32 rows x 128 bytes (this warp's box) and sends it with TMA.
      auto send_box = [&](const uint4 (&chunk)[8], int col) {
        // The box written two stores ago must have been read out by its TMA.
        if (lane == 0) bulk_wait_read_1();
        __syncwarp();
        uint8_t* box = stg + sb * 4096;
        stage_row(box, lane, chunk);
        fence_async_shared();
        __syncwarp();
        if (lane == 0) {
          if (bf16_out) tma_store_2d(&tmC, col, row_base, su32(box));
          else tma_reduce_add_2d(&tmC, col, row_base, su32(box));
          bulk_commit();
        }
        sb ^= 1;
      };
      // A split tile: add the other parts into this CTA's accumulator in TMEM first,
      // so the epilogue below is the same for every tile.
      if (finish && nparts > 1 && row_base < g.M) {
#pragma unroll 1
        for (int c = 0; c < BN; c += 32) {
          if (nt * BN + c >= g.N) break;
          uint32_t r[32];
          tmem_ld32(tbase + (uint32_t)c, r);
          combine32(c, r);
          tmem_st32(tbase + (uint32_t)c, r);
        }
        tmem_st_wait();
      }
      // 64 columns per step: both 32-column TMEM loads in flight under one wait.
#pragma unroll 1
      for (int c = 0; finish && c < BN; c += 64) {
        const int col0 = nt * BN + c;
        if (row_base >= g.M || col0 >= g.N) continue;  // uniform across the warp
        const bool two = c + 32 < BN && col0 + 32 < g.N;  // second 32-column half present
        // This step's bias (bf16 output) or bias and gate of the first half (fp32
        // output), requested before the TMEM loads so the two latencies overlap.
        float4 pb[8], pg[8];
        if (g.bias != nullptr) {
#pragma unroll
          for (int j = 0; j < 8; ++j)
            pb[j] = __ldg(reinterpret_cast<const float4*>(g.bias + col0) + (bf16_out ? 2 * j : j));
        }
        if (!bf16_out && g.epi == EPI_RESID_GATE) {
#pragma unroll
          for (int j = 0; j < 8; ++j) pg[j] = __ldg(reinterpret_cast<const float4*>(g.gate + col0) + j);
        }
        uint32_t r0[32], r1[32];
        tmem_ld32_nowait(tbase + (uint32_t)c, r0);
        if (two) tmem_ld32_nowait(tbase + (uint32_t)(c + 32), r1);
        tmem_ld_wait();
        uint4 chunk[8];
        if (bf16_out) {
          const bool gelu = g.epi == EPI_GELU;
#pragma unroll
          for (int j = 0; j < 8; ++j) {  // columns c + 8j .. c + 8j + 7 (bias in lane c/8 + j)
            float v[8];
#pragma unroll
            for (int e = 0; e < 8; ++e) v[e] = __uint_as_float(j < 4 ? r0[8 * j + e] : r1[8 * j + e - 32]);
            if (g.bias != nullptr) {
              const float4 b0 = pb[j];  // columns c + 8j .. c + 8j + 3 (first four of eight)
              const float4 b1 = __ldg(reinterpret_cast<const float4*>(g.bias + col0 + 8 * j + 4));
              v[0] += b0.x; v[1] += b0.y; v[2] += b0.z; v[3] += b0.w;
              v[4] += b1.x; v[5] += b1.y; v[6] += b1.z; v[7] += b1.w;
            }
            if (gelu) {
#pragma unroll
              for (int e = 0; e < 8; ++e) v[e] = gelu_tanh(v[e]);
            }
            chunk[j] = make_uint4(pack2(v[0], v[1]), pack2(v[2], v[3]), pack2(v[4], v[5]),
                                  pack2(v[6], v[7]));
          }
          send_box(chunk, col0);  // columns >= N are clipped by the tensor map
        } else {
          const bool gated = g.epi == EPI_RESID_GATE;
#pragma unroll
          for (int hh = 0; hh < 2; ++hh) {
            if (hh == 1 && !two) break;
            const uint32_t* r = hh == 0 ? r0 : r1;
            const int cc = c + 32 * hh;
#pragma unroll
            for (int j = 0; j < 8; ++j) {
              float4 v = make_float4(__uint_as_float(r[4 * j]), __uint_as_float(r[4 * j + 1]),
                                     __uint_as_float(r[4 * j + 2]), __uint_as_float(r[4 * j + 3]));
              const int cg = nt * BN + cc + 4 * j;  // columns cg .. cg + 3
              if (g.bias != nullptr) {
                const float4 b = hh == 0 ? pb[j] : __ldg(reinterpret_cast<const float4*>(g.bias + cg));
                v.x += b.x; v.y += b.y; v.z += b.z; v.w += b.w;
              }
              if (gated) {
                const float4 gg = hh == 0 ? pg[j] : __ldg(reinterpret_cast<const float4*>(g.gate + cg));
                v.x *= gg.x; v.y *= gg.y; v.z *= gg.z; v.w *= gg.w;
              }
              chunk[j] = make_uint4(__float_as_uint(v.x), __float_as_uint(v.y),
                                    __float_as_uint(v.z), __float_as_uint(v.w));
            }
            send_box(chunk, nt * BN + cc);
          }
        }
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

// CTAs of one kernel instantiation resident at once on the current device
// (one per SM: the kernel's shared memory admits no second).
int max_workers() { return num_sms(); }

std::atomic<int> g_gemm_raster{0};  // 0: the default rule above

template <int BN, int STAGES>
cudaError_t launch_tc(const void* A, const void* W, const GemmArgs& g_in, bool stream_k,
                      cudaStream_t s) {
  using S = TcShape<BN, STAGES>;
  GemmArgs g = g_in;
  g.raster = g_gemm_raster.load();
  if (g.raster <= 0) g.raster = RASTER_DEFAULT;
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
  const int m_units = (g.M + BM - 1) / BM;
  const int tiles = m_units * ((g.N + BN - 1) / BN);
  const int wmax = max_workers();
  int workers = tiles < wmax ? tiles : wmax;
  SkArgs sk = {nullptr, nullptr, 0, 0};
  if (stream_k) {
    // All but the last full wave and the partial one are taken whole and
    // round-robin (the tiles in flight stay neighbours in the raster order, so
    // their A and W blocks are shared in L2); stream-K evens out the rest.
    const int full = tiles / wmax;
    sk.dp_tiles = full > 1 ? (full - 1) * wmax : 0;
    sk.units = (int64_t)(tiles - sk.dp_tiles) * (g.K / BK);
    if (sk_scratch(s, (size_t)4 * tiles, (size_t)2 * wmax * BM * BN, &sk.cnt, &sk.ws))
      workers = wmax;
    else
      sk = {nullptr, nullptr, 0, 0};
  }
  count_launch();
  return launch_pdl(k_gemm_tc<BN, STAGES>, workers, 192, S::SMEM, s, ta, tb, tc, g, sk);
}

cudaError_t gemm_dispatch(const void* A, const void* W, const GemmArgs& g, int sched,
                          cudaStream_t s) {
  // Schedule and tile width by a makespan model: every worker of a wave runs
  // concurrently, so a data-parallel launch costs about rounds x k-blocks x
  // (BN + 150), the 150 columns' worth of per-k-block overhead fitted to
  // measured tile times (a 192-wide tile takes about 0.85x the time of a
  // 256-wide one).  Ties go to the wider tile.  Stream-K with 256-wide tiles
  // costs the average number of work tiles per worker (fractional) times the
  // same figure, plus SK_FIXUP; it is taken only when no tile spans more than
  // SK_MAX_PARTS workers.
  const int m_units = (g.M + BM - 1) / BM;
  const bool fp32_out = g.epi == EPI_RESID || g.epi == EPI_RESID_GATE;  // 32-column epilogue chunks
  const long nk = g.K / BK;
  int best_bn = 256;
  long best_cost = -1;
  for (int bn : {256, 192, 160, 128}) {
    if (bn == 160 && !fp32_out) continue;  // bf16 epilogue chunks are 64 columns wide
    const int wk = max_workers();
    const long tiles = (long)m_units * ((g.N + bn - 1) / bn);
    const long cost = ((tiles + wk - 1) / wk) * nk * (bn + 150);
    if (best_cost < 0 || cost < best_cost) {
      best_cost = cost;
      best_bn = bn;
    }
  }
  if (sched != 1) {
    const int wk = max_workers();
    const long tiles = (long)m_units * ((g.N + 255) / 256);
    const long units = tiles * nk, per_worker = units / wk;
    const bool spans_ok =
        per_worker > 0 && 1 + (nk - 1 + per_worker - 1) / per_worker <= SK_MAX_PARTS;
    const double sk_cost = (double)tiles / wk * nk * (256 + 150) + SK_FIXUP;
    if (spans_ok && (sched == 2 || (tiles > wk / 2 && sk_cost < (double)best_cost)))
      return launch_tc<256, 4>(A, W, g, true, s);
  }
  if (best_bn == 256) return launch_tc<256, 4>(A, W, g, false, s);
  if (best_bn == 192) return launch_tc<192, 4>(A, W, g, false, s);
  if (best_bn == 160) return launch_tc<160, 5>(A, W, g, false, s);
  return launch_tc<128, 6>(A, W, g, false, s);
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

namespace {
// Stream-K counters and partial-sum slots, one set per (device, stream): the
// kernels of one stream run one after another and leave every counter at zero,
// so the GEMM and attention launches of a stream share them.
struct SkScratch {
  int* cnt = nullptr;
  size_t ncnt = 0;
  float* ws = nullptr;
  size_t nws = 0;
};
std::mutex g_sk_mu;
std::map<std::pair<int, cudaStream_t>, SkScratch> g_sk;
std::atomic<uint64_t> g_sk_gen{0};
}  // namespace

uint64_t sk_scratch_generation() { return g_sk_gen.load(); }

bool sk_scratch(cudaStream_t s, size_t ncnt, size_t nws, int** cnt, float** ws) {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return false;
  std::lock_guard<std::mutex> lk(g_sk_mu);
  SkScratch& sc = g_sk[std::make_pair(dev, s)];
  if (sc.ncnt < ncnt || sc.nws < nws) {
    g_sk_gen.fetch_add(1);
    if (cudaStreamSynchronize(s) != cudaSuccess) return false;
    cudaFree(sc.cnt);
    cudaFree(sc.ws);
    sc = SkScratch();
    const size_t nc = ncnt > 4096 ? ncnt : 4096, nw = nws;
    if (dev_malloc((void**)&sc.cnt, nc * sizeof(int)) != cudaSuccess ||
        dev_malloc((void**)&sc.ws, nw * sizeof(float)) != cudaSuccess ||
        cudaMemsetAsync(sc.cnt, 0, nc * sizeof(int), s) != cudaSuccess) {
      cudaGetLastError();
      cudaFree(sc.cnt);
      cudaFree(sc.ws);
      sc = SkScratch();
      return false;
    }
    sc.ncnt = nc;
    sc.nws = nw;
  }
  *cnt = sc.cnt;
  *ws = sc.ws;
  return true;
}


namespace {
std::atomic<int> g_schedule{0};
}

void set_gemm_schedule(int mode) { g_schedule.store(mode); }

namespace {
__global__ void k_wait_selftest(int* err, long long limit, int code) {
  __shared__ uint64_t bar;
  __shared__ int abort_flag;
  if (threadIdx.x == 0) {
    mbar_init(su32(&bar), 1);
    abort_flag = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  __syncthreads();
  // Nothing arrives on the barrier: its phase 0 never completes.
  if (threadIdx.x == 0) mbar_wait(su32(&bar), 0, &abort_flag, err, code, limit);
}
}  // namespace

cudaError_t wait_selftest(int* err, long long limit, int code, cudaStream_t s) {
  k_wait_selftest<<<1, 32, 0, s>>>(err, limit, code);
  count_launch();
  return cudaGetLastError();
}
void set_gemm_raster(int group) { g_gemm_raster.store(group > 0 ? group : 0); }

cudaError_t gemm_bf16_tc(const void* A, const void* W, const GemmArgs& g, cudaStream_t s) {
  if (g.M <= 0 || g.N <= 0) return cudaSuccess;
  if (g.K <= 0 || g.K % BK != 0 || g.N % 32 != 0 || g.ldo % 8 != 0) return cudaErrorInvalidValue;
  if ((((uintptr_t)A) | ((uintptr_t)W) | ((uintptr_t)g.out)) & 15) return cudaErrorMisalignedAddress;
  if (g.bias != nullptr && (((uintptr_t)g.bias) & 15)) return cudaErrorMisalignedAddress;
  if (g.epi == EPI_RESID_GATE && (g.gate == nullptr || (((uintptr_t)g.gate) & 15)))
    return cudaErrorInvalidValue;
  return gemm_dispatch(A, W, g, g_schedule.load(), s);
}

}  // namespace track
