// Internal declarations shared by the CUDA translation units of libtrack.
// Kernel launchers take device pointers and a stream and return cudaError_t.
#pragma once

#include <cuda_runtime.h>
#include <stdint.h>

#include <utility>

namespace track {

// Programmatic dependent launch: a kernel launched this way may start while the
// previous kernel on its stream is still running; it calls pdl_wait() before it
// touches global memory that kernel reads or writes, and pdl_release() to let the
// next kernel start the same way.
__device__ __forceinline__ void pdl_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }
__device__ __forceinline__ void pdl_release() {
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
}

template <typename... KArgs, typename... Args>
cudaError_t launch_pdl(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem,
                       cudaStream_t s, Args&&... args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, kernel, std::forward<Args>(args)...);
}

enum Dtype { F32 = 0, BF16 = 1 };
enum Epi { EPI_STORE = 0, EPI_GELU = 1, EPI_RESID_GATE = 2, EPI_RESID = 3 };

// Error word written by kernels whose pipeline waits ran out (0 = none).
// One per device, zeroed at first use; read and cleared by track_sync.
int* device_error_word();

// Counts every kernel launch made by the library.
void count_launch(int n = 1);

// Records msg as this thread's last error (returned by track_last_error); returns code.
int report_error(int code, const char* msg);

// ---------------------------------------------------------------- GEMM
struct GemmArgs {
  int M, N, K;
  int epi;             // Epi
  const float* bias;   // [N] or nullptr
  const float* gate;   // [N] (EPI_RESID_GATE)
  void* out;           // T [M, ldo] (STORE/GELU) or fp32 [M, ldo] (RESID*)
  int ldo;
  int* err;            // device error word
  int raster;          // bf16 tensor-core GEMM: row units per raster group (set by its launcher)
  int w_static = 0;    // W is never written by a kernel (model weights): it may be
                       // requested before the grid dependency wait
};

// fp32 FFMA GEMM: out = A[M,K] . W[N,K]^T (+ epilogue), all fp32.
cudaError_t gemm_f32(const float* A, const float* W, const GemmArgs& g, cudaStream_t s);
// Row units per raster group of the bf16 tensor-core GEMM (0: the default).
void set_gemm_raster(int group);
// Device allocation of the library's own buffers (weights, workspaces,
// scratch); fails like an exhausted device while track_fail_next_allocations
// has failures pending.
cudaError_t dev_malloc(void** p, size_t bytes);
void set_failing_allocations(int n);
// One CTA waits, through the tensor-core kernels' bounded mbarrier wait, on a
// barrier nothing completes; after `limit` SM cycles the wait gives up and
// records `code` in the device error word.
cudaError_t wait_selftest(int* err, long long limit, int code, cudaStream_t s);

// bf16 tcgen05 GEMM: A bf16 [M,K] and W bf16 [N,K], fp32 accumulation in TMEM.
// Requires K % 64 == 0, N % 32 == 0 and 16-byte aligned A, W and out.
cudaError_t gemm_bf16_tc(const void* A, const void* W, const GemmArgs& g, cudaStream_t s);
// Stream-K counters (zero between launches) and fp32 partial-sum slots of the
// stream, grown on demand (a growth synchronizes the stream).  False if they
// cannot be allocated.
bool sk_scratch(cudaStream_t s, size_t ncnt, size_t nws, int** cnt, float** ws);
// Bumped whenever any stream-K scratch is reallocated (recorded graphs hold its addresses).
uint64_t sk_scratch_generation();
// 0 auto, 1 data-parallel, 2 stream-K where the shape allows it.
void set_gemm_schedule(int mode);

// ---------------------------------------------------------------- attention
// One attention operand: element (s, h, l, e) of its [S, H, L, hd] view lives at
// ptr + s*ss + h*hs + l*ls + e (strides in elements).  Head-major buffers have
// ls = hd, hs = L*hd; token-major projection outputs [S*L, ld] with head h at
// columns h*hd have ls = ld, hs = hd.
struct AttnOperand {
  const void* ptr;
  int64_t ls, hs, ss;
};
inline AttnOperand head_major(const void* p, int H, int L, int hd) {
  return {p, hd, (int64_t)L * hd, (int64_t)H * L * hd};
}
inline AttnOperand token_major(const void* p, int L, int ld, int hd) {
  return {p, ld, hd, (int64_t)L * ld};
}
// O [S, Lq, H, hd] (token-major) = softmax(Q K^T / sqrt(hd)) V.
cudaError_t attention_f32(const AttnOperand& Q, const AttnOperand& K, const AttnOperand& V,
                          float* O, int S, int H, int Lq, int Lk, int hd, cudaStream_t s);
// 0 auto, 1 data-parallel, 2 stream-K where the shape allows it.
void set_attention_schedule(int mode);
cudaError_t attention_bf16(const AttnOperand& Q, const AttnOperand& K, const AttnOperand& V,
                           void* O, int S, int H, int Lq, int Lk, int hd, cudaStream_t s);

// ---------------------------------------------------------------- elementwise
cudaError_t convert_f32(const float* src, void* dst, int dtype, int64_t n, cudaStream_t s);
cudaError_t seed_fill(void* dst, int dtype, uint64_t state, int64_t n, float scale,
                      float offset, int has_offset, cudaStream_t s);
// emb[freq_dim] = [cos(t f_i), sin(t f_i)], f_i = 10000^(-i/(freq_dim/2)) (double precision)
cudaError_t sinusoid(float t, float* emb, int freq_dim, cudaStream_t s);
// out[r] = b[r] + sum_k W[r,k] * act(in[k]); act = SiLU if silu_in else identity
cudaError_t matvec(const void* W, int dtype, const float* in, const float* b, float* out, int rows,
                   int cols, int silu_in, cudaStream_t s);
// mod_all[l,6,d] = e0[6,d] + mod_bias[l,6,d];  head_mod[2,d] = e[d] + head_bias[2,d]
cudaError_t modulation(const float* e0, const float* mod_bias, int layers, const float* e,
                       const float* head_bias, int d, float* mod_all, float* head_mod,
                       cudaStream_t s);
// x_res[s*L + tok, :] = patch(x[s % B], tok) . W_pe^T + b_pe
cudaError_t patch_embed(const float* x, int B, int nseq, int C, int F, int H, int W,
                        const void* Wpe, int dtype, const float* bpe, int d, float* xres,
                        cudaStream_t s);
// out = LN(x) * (1 + scale) + shift (mode 0) or LN(x) * g + b (mode 1); out in dtype
cudaError_t ln_modulate(const float* x, int M, int d, const float* a, const float* b, int mode,
                        float eps, void* out, int dtype, cudaStream_t s);
// In place on a token-major buffer [rows, ld] (row r = token r % L of sequence
// r / L): for each of nsec sections of d columns, section j at column
// off0 + j*off_stride with gain gain0 + j*gain_stride: RMSNorm over the d values
// times the gain, then (rope) the 3D rotary embedding of every head of hd.
struct NormRopeArgs {
  void* buf; int ld; int rows; int L; int hd; int d;
  int nsec; int64_t off0, off_stride;
  const float* gain0; int64_t gain_stride;
  int rope;
  const float2* rope_tab;   // per-axis (cos, sin) tables, see build_rope_table
  int Fp, Hp, Wp;
  float eps;
  int dtype;
};
cudaError_t qk_norm_rope(const NormRopeArgs& a, cudaStream_t s);
// Head: LN(x)*(1+scale)+shift, . head_W^T + head_b, unpatchify into out [nseq, C, F, H, W]
cudaError_t head_unpatchify(const float* xres, int nseq, int L, int d, const float* head_mod,
                            const void* Whead, int dtype, const float* bhead, float eps, int C,
                            int F, int H, int W, float* out, cudaStream_t s);
// Token-major [nseq * L, 4C] -> [nseq, C, F, H, W] (exact inverse of patchify).
cudaError_t unpatchify(const float* tokv, int nseq, int L, int C, int F, int H, int W, float* out,
                       cudaStream_t s);
// Eq. 1 and Eq. 2 on n floats.
cudaError_t cfg_combine(const float* fc, const float* fu, int64_t n, float w, float* p,
                        cudaStream_t s);
cudaError_t euler_step(float* x, const float* v, int64_t n, float dsig, cudaStream_t s);
// Step i of the second-order predictor-corrector scheduler (Eq. 2 with history):
// x (the latent the model saw) becomes x_{i+1}; (xc, vp) is the history,
// read for i > 0 and rewritten.  sigmas: host.
cudaError_t multistep_step(float* x, const float* v, float* xc, float* vp, int64_t n,
                           const float* sigmas, int i, cudaStream_t s);
cudaError_t cfg_euler(float* x, const float* fc, const float* fu, int64_t n, float w, float dsig,
                      cudaStream_t s);
// Sec. 4.4 frequency-band split of Eq. 4 (see bands.cu): out [B, 6] device fp32;
// scratch holds band_scratch_floats(B, C, F, H, W) floats.
size_t band_scratch_floats(int B, int C, int F, int H, int W);
cudaError_t band_disagreement(const float* vL, const float* vS, int B, int C, int F, int H, int W,
                              float eps, float* out, float* scratch, cudaStream_t s);

// Eq. 4: partial sums then a fixed-order final combine; scratch holds B*nblk*2 floats.
int disagreement_blocks(int64_t n_per_sample, int B);
cudaError_t disagreement(const float* vL, const float* vS, int B, int64_t n, float eps,
                         float* accum, float* scratch, int nblk, cudaStream_t s);
// The same computation (same bits) in one launch; counters: B ints, zero before
// the call, left at zero by it.  With x non-null the same pass also applies the
// Euler update x[b] += dsig * vL[b] (x must not alias vL or vS).
cudaError_t disagreement_fused(const float* vL, const float* vS, int B, int64_t n, float eps,
                               float* accum, float* scratch, int* counters, int nblk,
                               cudaStream_t s, float* x = nullptr, float dsig = 0.f);

int num_sms();

}  // namespace track
