/*
 * track.h - C ABI of the GB300 (sm_103a) implementation of TRACK's routed
 * denoising hot path ("Accelerating Video Diffusion via Training-Free
 * Trajectory Routing").
 *
 * Conventions for every entry point:
 *  - Every function returns an int status (TRACK_OK = 0 or a TRACK_E* code)
 *    unless stated otherwise.  No function aborts, prints or throws; the text
 *    of the last error on the calling thread is returned by track_last_error().
 *  - "device" pointers are CUDA device memory owned by the caller, 16-byte
 *    aligned, and are read/written in stream order on the given stream
 *    (a cudaStream_t passed as void*; NULL means the legacy default stream).
 *    Calls return once the work is enqueued; asynchronous device errors
 *    surface at the next call that synchronizes, or at track_sync().
 *  - "host" pointers are ordinary host memory, read/written before return.
 *  - Latents are fp32 [B, C, F, H, W] (C = 16), contiguous.  Text
 *    conditioning is fp32 [B, Lt, Dtxt], contiguous.
 *  - Models with dtype TRACK_BF16 keep weight matrices and activations in
 *    bf16 and accumulate in fp32 on the tensor cores; TRACK_FP32 models run
 *    true fp32 (FFMA) arithmetic throughout (no TF32).
 */
#ifndef TRACK_H
#define TRACK_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* ---- status codes ------------------------------------------------------ */
#define TRACK_OK 0
#define TRACK_EINVAL 1       /* bad argument (NULL, shape, range, NaN score ...) */
#define TRACK_ENOMEM 2       /* device or host allocation failed */
#define TRACK_ECUDA 3        /* a CUDA runtime/driver call failed */
#define TRACK_EUNSUPPORTED 4 /* valid request this build does not support */
#define TRACK_ETIMEOUT 5     /* a device pipeline wait ran out (kernel gave up) */

#define TRACK_FP32 0
#define TRACK_BF16 1

/* Epilogues of track_linear (Y = X W^T + b, then): */
#define TRACK_EPI_STORE 0      /* Y stored in the model dtype                     */
#define TRACK_EPI_GELU 1       /* GELU_tanh(Y) stored in the model dtype          */
#define TRACK_EPI_RESID_GATE 2 /* fp32 R[m,n] += gate[n] * Y[m,n]                 */
#define TRACK_EPI_RESID 3      /* fp32 R[m,n] += Y[m,n]                           */

typedef void* track_stream; /* a cudaStream_t */

/*
 * Architecture of one denoiser f_m (the black box of Eq. 1).  The paper fixes
 * no internals (Sec. 3.1, "Compatible model pairs": the pair shares latent,
 * output shape, conditioning interface and prediction target; architectures
 * may differ).  This library implements a Wan-style video DiT: patch 1x2x2,
 * adaLN-modulated self-attention with 3D RoPE and RMSNorm(q, k) over the model
 * width, cross-attention to the projected text, GELU_tanh MLP, modulated head.
 * Requirements: dim % heads == 0, head_dim = dim/heads in {64, 128},
 * in_ch * 4 == 64, frames/height/width divisible by the patch, dim, ffn and
 * text_dim multiples of 64, freq_dim == 256.
 */
typedef struct track_arch {
  int dim;      /* model width d                      */
  int layers;   /* transformer blocks                 */
  int heads;    /* attention heads                    */
  int ffn;      /* MLP hidden width                   */
  int text_dim; /* Dtxt, width of the text input      */
  int text_len; /* Lt, text tokens per sample         */
  int in_ch;    /* latent channels C (16)             */
  int frames;   /* latent F                           */
  int height;   /* latent H                           */
  int width;    /* latent W                           */
  int patch_f, patch_h, patch_w; /* must be 1, 2, 2   */
  int freq_dim; /* timestep sinusoid width (256)      */
  int dtype;    /* TRACK_FP32 or TRACK_BF16           */
  float eps;    /* LayerNorm / RMSNorm epsilon (1e-6) */
} track_arch;

typedef struct track_model track_model;

/* ---- library ----------------------------------------------------------- */

/* Text of the last error on this thread ("" if none).  Never NULL. */
const char* track_last_error(void);

/* ABI version of this header (returns the integer, not a status). */
int track_abi_version(void);

/* Waits for all work on stream s and reports device-side errors: TRACK_ECUDA
 * for a CUDA error, TRACK_ETIMEOUT if a kernel abandoned a pipeline wait
 * (the flag is cleared by this call). */
int track_sync(track_stream s);

/* Number of kernels this library has launched since load (returns the count). */
int64_t track_launch_count(void);

/* Failure detection, exercised without a GPU fault.
 *
 * track_wait_selftest launches one CTA whose thread waits, through the same
 * bounded mbarrier wait every tensor-core kernel uses for its pipeline, on a
 * barrier that nothing completes.  After limit_cycles SM cycles the wait gives
 * up: the CTA records TRACK_WAIT_SELFTEST_CODE in the device error word and
 * exits, and the context stays usable.  Returns TRACK_OK once launched on s;
 * the next track_sync on s then returns TRACK_ETIMEOUT naming that code and
 * clears the word.  EINVAL unless 1e3 <= limit_cycles <= 2e9 (the kernels'
 * own limit is 2e9 cycles, about one second).
 *
 * track_fail_next_allocations makes the next n device allocations the library
 * makes for itself (weights, workspaces, scratch) fail as if the device were
 * out of memory: the call that needed one returns TRACK_ENOMEM, or, where a
 * fallback exists (stream-K scratch), takes it.  n = 0 clears pending
 * failures; EINVAL for n < 0. */
#define TRACK_WAIT_SELFTEST_CODE 99
int track_wait_selftest(int64_t limit_cycles, track_stream s);
int track_fail_next_allocations(int n);

/* Kernel timing: while enabled, the GEMM, attention, normalization, update
 * and Eq. 4 launches inside track_denoise/track_denoise_step/track_calibrate/
 * track_sample are bracketed by CUDA events on their stream.
 * track_profile_read synchronizes those events and returns, per class (0 =
 * GEMM, 1 = self-attention, 2 = LayerNorm-modulate, 3 = RMSNorm of q/k with
 * RoPE, 4 = guidance combine and scheduler update, 5 = Eq. 4 reduction (in
 * track_calibrate fused with the trajectory's Euler update), 6 =
 * cross-attention), the summed event time in ms, the summed algorithmic work
 * (FLOPs for classes 0, 1 and 6, bytes moved for the others) and the number of launches, then clears the
 * records.  Arrays are host, length TRACK_PROFILE_CLASSES.  In a graph
 * recorded by track_sample_graph while timing is enabled, the brackets are
 * event-record nodes of the graph: each replay re-records the same events, so
 * read after every replay. */
#define TRACK_PROFILE_CLASSES 7
int track_profile_enable(int enable);
int track_profile_read(double* ms, double* flops, int64_t* launches);

/* ---- models (Sec. 3.1 "Compatible model pairs") --------------------------- */

/* Number of canonical weight tensors of arch (returns the count, or -1). */
int track_weight_count(const track_arch* arch);

/* Shape of canonical tensor `index` (rows, cols; cols = 1 for vectors).
 * Canonical order: pe.W[d,64] pe.b[d] txt.W1[d,Dtxt] txt.b1 txt.W2[d,d] txt.b2
 * tim.W1[d,256] tim.b1 tim.W2[d,d] tim.b2 mod.W[6d,d] mod.b[6d]; per block:
 * mod_bias[6,d] q.W[d,d] q.b k.W k.b v.W v.b o.W o.b qn.g kn.g ln3.g ln3.b
 * cq.W cq.b ck.W ck.b cv.W cv.b co.W co.b cqn.g ckn.g ffn.W1[F,d] ffn.b1[F]
 * ffn.W2[d,F] ffn.b2[d]; then head_bias[2,d] head.W[64,d] head.b[64].
 * Matrices are [out, in] row-major. */
int track_weight_shape(const track_arch* arch, int index, int64_t* rows, int64_t* cols);

/* Creates a model on the current CUDA device from host fp32 weights.
 * weights[i] points to canonical tensor i (track_weight_count entries).  The
 * library copies (and, for TRACK_BF16, rounds to nearest-even bf16) every
 * matrix into device memory it owns; the caller may free the host arrays
 * after return.  Synchronous.  EINVAL for an unsupported arch. */
int track_model_create(const track_arch* arch, const float* const* weights, track_model** out);

/* Same, with weights generated on the device by the library's counter-based
 * generator (SplitMix64 stream per (seed, tensor index); approximately normal
 * Irwin-Hall-4 draws; matrices N(0, 1/fan_in), biases N(0, 0.02^2), norm gains
 * 1 + N(0, 0.05^2), LayerNorm offsets N(0, 0.05^2)).  The values are bit-for-bit
 * those the repository's host generator produces for the same seed. */
int track_model_create_seeded(const track_arch* arch, uint32_t seed, track_model** out);

int track_model_destroy(track_model* m);

/* Sec. 3.1: 1 if a and b can be interchanged within one trajectory (same
 * latent shape, text interface and patch), 0 if not, negative on error. */
int track_models_compatible(const track_model* a, const track_model* b);

/* Drops the model's cache of projected text conditioning.  track_denoise
 * caches the text projection and the per-block cross-attention keys/values
 * keyed on the (cond, uncond, B) pointers it was last given; call this when
 * the data behind the same pointers changes. */
int track_invalidate_ctx(track_model* m);

/* ---- denoiser and guidance (Eq. 1) --------------------------------------- */

/* v_out = p_m(x_t, t) of Eq. 1 for B samples at model timestep t:
 *   f(x_t, t, uncond) + cfg_scale * (f(x_t, t, cond) - f(x_t, t, uncond)).
 * x_t, v_out: device fp32 [B, C, F, H, W]; cond, uncond: device fp32
 * [B, Lt, Dtxt].  With cfg_scale == 1 the unconditional pass is skipped, v_out
 * equals f(x_t, t, cond) exactly and uncond may be NULL (else EINVAL).
 * cond and uncond are batched into one forward of 2B sequences.  v_out must
 * not alias x_t.  The first call at a new B grows the model's workspace
 * (cudaMalloc, synchronizing). */
int track_denoise(track_model* m, const float* x_t, int B, float t, const float* cond,
                  const float* uncond, float cfg_scale, float* v_out, track_stream s);

/* One scheduler step with this denoiser (Eq. 2/Eq. 3 with the flow-matching
 * Euler update): evaluates the model at t = 1000 * sigma_t and updates x in
 * place, x += (sigma_next - sigma_t) * p, with the guidance combine fused into
 * the update kernel. */
int track_denoise_step(track_model* m, float* x, int B, float sigma_t, float sigma_next,
                       const float* cond, const float* uncond, float cfg_scale, track_stream s);

/* Eq. 1 combine on n elements: p = f_u + w * (f_c - f_u) (p = f_c if w == 1). */
int track_cfg(const float* f_c, const float* f_u, int64_t n, float w, float* p_out,
              track_stream s);

/* ---- scheduler (Eq. 2, flow-matching Euler instance) ---------------------- */

/* sigmas_out (host, n_steps + 1 floats): sigma_i = s*u/(1+(s-1)*u), u = 1 - i/N,
 * computed in double and rounded to float; sigma_0 = 1, sigma_N = 0.  The
 * model timestep of step i is t_i = 1000 * sigma_i. */
int track_schedule(int n_steps, float shift, float* sigmas_out);

/* In place x += (sigma_next - sigma_t) * v on n device floats (Eq. 2). */
int track_step(float* x_t, const float* v, int64_t n, float sigma_t, float sigma_next,
               track_stream s);

/* Fused Eq. 1 + Eq. 2: x += (sigma_next - sigma_t) * (f_u + w (f_c - f_u)).
 * f_u may be NULL when w == 1 (then p = f_c). */
int track_cfg_step(float* x, const float* f_c, const float* f_u, int64_t n, float w,
                   float sigma_t, float sigma_next, track_stream s);

/* ---- calibration score (Eq. 4, Eq. 5) ------------------------------------ */

/* Eq. 4 per sample b: r_b = ||v_S[b] - v_L[b]||_2 / max(||v_L[b]||_2, eps), norms
 * over the n_per_sample elements of sample b; adds r_b to score_accum[b]
 * (device, B floats).  Deterministic: identical inputs give bitwise-identical
 * results (fixed-order two-level reduction, no floating-point atomics).
 * Uses library-owned device scratch per (device, stream); s must be a stream
 * of the current device. */
int track_disagreement(const float* v_L, const float* v_S, int B, int64_t n_per_sample,
                       float eps, float* score_accum, track_stream s);

/* One step of the calibration trajectory after both predictions (Sec. 3.2.1):
 * adds Eq. 4's r_b of (v_L, v_S) to score_accum[b] exactly as
 * track_disagreement does (same bits), and advances the trajectory by the large
 * model's prediction, x[b] += (sigma_next - sigma_t) * v_L[b] (Eq. 2, Euler,
 * the bits of track_step), in one pass that reads v_L once for both.
 * x: device fp32 [B, n_per_sample], in/out, must not overlap v_L or v_S
 * (EINVAL).  Same scratch, stream and determinism rules as track_disagreement. */
int track_disagreement_update(const float* v_L, const float* v_S, int B, int64_t n_per_sample,
                              float eps, float* score_accum, float* x, float sigma_t,
                              float sigma_next, track_stream s);

/* Eq. 5 on the host: q[k] = (1/M) sum_j r[j*N + k] (r host [M, N]), summed in j
 * order in double and rounded to float. */
int track_mean_score(const float* r, int M, int N, float* q_out);

/* The offline artifact of calibration (Sec. 3.2.1): the per-sample, per-step
 * disagreement map r [M, N] (host, row j = calibration sample j) and its mean
 * q [N] (Eq. 5), in a file, so that the policy can be rebuilt without the
 * models and calibration resumed sample by sample (rows are independent:
 * load, calibrate further samples, append their rows, save).  Format, all
 * little-endian: 8 bytes "TRKSCORE", uint32 version (1), uint32 M, uint32 N,
 * uint64 config_hash (the caller's identifier of the model pair, schedule and
 * CFG scale), float32 r[M*N] row-major, float32 q[N] as track_mean_score
 * computes it.
 *
 * track_score_map_save writes (replaces) path; EINVAL for bad arguments, a
 * negative or NaN score, or a file that cannot be written.  track_score_map_load reads path into r (capacity r_cap floats) and
 * q (capacity q_cap floats; q may be NULL), and sets *M, *N and *config_hash;
 * EINVAL if the file is missing, truncated, has another magic or version, or
 * does not fit the capacities.  Host only. */
int track_score_map_save(const char* path, const float* r, int M, int N, uint64_t config_hash);
int track_score_map_load(const char* path, float* r, int64_t r_cap, float* q, int64_t q_cap,
                         int* M, int* N, uint64_t* config_hash);

/* ---- policy (Eq. 6, Eq. 7, top-K switching of Sec. 3.2.3) ------------------ */

/* policy_out[k] = 1 (small model) for the K steps with the lowest score, else
 * 0 (large model).  Ranking is on the fp32 score; ties at the K/K+1 boundary
 * go to the lower step index.  EINVAL if K < 0, K > N, N < 1 or any score is
 * NaN or negative.  Host only, bit-exact. */
int track_policy_topk(const float* score_map, int N, int K, uint8_t* policy_out);

/* Equal-budget baseline policies of the paper's ablation (Sec. 4.5, Table 2):
 * each routes exactly K of the N steps to the small model (policy_out[k] = 1).
 * First-K: steps 0..K-1.  Last-K: steps N-K..N-1.  Random-K: a uniformly random
 * K-subset by a partial Fisher-Yates shuffle of 0..N-1, whose i-th swap partner
 * is i + (u_i mod (N - i)), u_i the i-th output of the SplitMix64 stream started
 * at state mix64(seed) (u_i = mix64(state + (i + 1) * 0x9E3779B97F4A7C15)).
 * EINVAL if N < 1 or K outside [0, N].  Host only, bit-exact. */
int track_policy_first_k(int N, int K, uint8_t* policy_out);
int track_policy_last_k(int N, int K, uint8_t* policy_out);
int track_policy_random_k(int N, int K, uint64_t seed, uint8_t* policy_out);

/* ---- loops (Sec. 3.2.1 calibration, Eq. 3 routed sampling) ---------------- */

/* Reference-trajectory calibration for B samples: for k in 0..n_steps-1,
 * p_L = track_denoise(L), p_S = track_denoise(S) on the same x, then
 * r_out[k*B + b] = Eq. 4 score, then x += (sigma_{k+1} - sigma_k) * p_L.
 * x: device [B, ...] in/out (ends as the all-large sample); sigmas: host
 * (n_steps + 1); r_out: device fp32 [n_steps, B] (overwritten). */
int track_calibrate(track_model* large, track_model* small, float* x, int B, const float* cond,
                    const float* uncond, float cfg_scale, const float* sigmas, int n_steps,
                    float eps, float* r_out, track_stream s);

/* Eq. 3: for i in 0..n_steps-1, the model policy[i] (0 = large, 1 = small)
 * supplies p and x += (sigma_{i+1} - sigma_i) * p; exactly one model per step.
 * policy, sigmas: host; x: device in/out. */
int track_sample(track_model* large, track_model* small, const uint8_t* policy,
                 const float* sigmas, int n_steps, float* x, int B, const float* cond,
                 const float* uncond, float cfg_scale, track_stream s);

/* Sec. 4.4: Eq. 4's disagreement split over frequency bands.  For each sample
 * b, D = v_S - v_L ([C, F, H, W], fp32) is transformed by the orthonormal 3-D
 * DFT over (F, H, W) per channel, and every bin's energy |D^|^2 goes to one
 * spatial band (radius of the (h, w) frequency in units of Nyquist:
 * low < 1/3 <= mid < 2/3 <= high) and one temporal band (|f| frequency in
 * units of Nyquist, same thirds); the paper gives no band edges, these are the
 * reading used.  bands_out[b * 6 + j] = sqrt(E_j) / max(||v_L[b]||, eps):
 * j = 0..2 spatial low/mid/high, 3..5 temporal low/mid/high (each triple's
 * squares add up to r^2 of Eq. 4).  v_L, v_S: device fp32 [B, C, F, H, W];
 * bands_out: device fp32 [B, 6], overwritten.  Deterministic.  Uses scratch
 * the library keeps per stream (4 B C F H W floats plus partials).
 * EUNSUPPORTED for an axis longer than 512. */
int track_band_disagreement(const float* v_L, const float* v_S, int B, int C, int F, int H, int W,
                            float eps, float* bands_out, track_stream s);

/* Eq. 2 with a scheduler history h_i (Sec. 3.1 allows any multistep solver and
 * TRACK keeps its state evolution unchanged across model switches): one step
 * of the second-order predictor-corrector for dx/dsigma = v.  With
 * h_i = sigmas[i+1] - sigmas[i] and r = h_i / h_{i-1}:
 *   i = 0:  xc = x,                                x <- xc + h_i v
 *   i > 0:  xc = xc' + (h_{i-1}/2) (v' + v),       x <- xc + h_i ((1 + r/2) v - (r/2) v')
 * where (xc', v') is the history from step i-1; then the history becomes
 * (xc, v).  x: device fp32 [n] in/out (in: the latent the model saw at step
 * i, out: the next one); v: device fp32 [n], the guided prediction made at x;
 * state: device fp32 [2 n], the corrected latent then the previous velocity,
 * caller-owned, read only for i > 0.  sigmas: host (n_steps + 1).  EINVAL for
 * i outside [0, n_steps) or v aliasing x or state.  The paper gives no
 * formulas for its pipelines' UniPC sampler; this scheme is the reading used. */
int track_multistep_step(float* x, const float* v, float* state, int64_t n, const float* sigmas,
                         int n_steps, int i, track_stream s);

/* Eq. 3 over the multistep scheduler of track_multistep_step: policy[i] picks
 * the model for step i, and the history runs through switches untouched.
 * state: device fp32 [2, B, C, F, H, W] scratch, caller-owned (contents on
 * entry ignored; on return, the history after the last step). */
int track_sample_multistep(track_model* large, track_model* small, const uint8_t* policy,
                           const float* sigmas, int n_steps, float* x, int B, const float* cond,
                           const float* uncond, float cfg_scale, float* state, track_stream s);

/* track_sample through a CUDA graph.  It computes the same values bit for bit,
 * with the text projection of cond/uncond recomputed on every call.  The
 * library keeps up to 32 recorded graphs, keyed by every argument (models,
 * policy and sigma values, pointers, B, cfg_scale, stream).  The first call
 * with a key runs eagerly and sizes every buffer the graph will address.  The
 * second call records the loop on s and instantiates it.  Later calls replay
 * it with one launch, so host launch time no longer paces the GPU.  Replays
 * read the current contents of x, cond and uncond.  A graph is dropped when
 * a model it uses is destroyed or a buffer it addresses is reallocated.
 * s must be a created stream: EINVAL for the legacy default stream (it cannot
 * be recorded).  Whether kernel timing (track_profile_enable) is on is part
 * of the key: a graph recorded with timing on carries an event-record node
 * before and after each GEMM, attention and normalization kernel (it runs the
 * same kernels, without the launch overlap that PDL gives between them), and
 * one recorded with timing off carries none.  This is a host-side mechanism;
 * the paper has no counterpart. */
int track_sample_graph(track_model* large, track_model* small, const uint8_t* policy,
                       const float* sigmas, int n_steps, float* x, int B, const float* cond,
                       const float* uncond, float cfg_scale, track_stream s);

/* ---- building blocks (the denoiser's kernels, for tests and benchmarks) --- */

/* Y = X W^T + bias with an epilogue (TRACK_EPI_*).  dtype selects the kernel:
 * TRACK_BF16 -> tcgen05 tensor-core GEMM (X bf16 [M,K], W bf16 [N,K], Y bf16
 * or fp32 residual), TRACK_FP32 -> FFMA GEMM (all fp32).  out has leading
 * dimension ldo (elements).  gate: fp32 [N] (RESID_GATE only); bias may be
 * NULL.  Requires K % 64 == 0 and N % 32 == 0 for TRACK_BF16. */
int track_linear(int dtype, const void* X, const void* W, const float* bias, int M, int N,
                 int K, int epilogue, const float* gate, void* out, int ldo, track_stream s);

/* Schedule of the TRACK_BF16 GEMM (process-wide, every device and stream).
 * TRACK_GEMM_AUTO (the default) picks per launch, by a makespan model, between
 * data-parallel (each CTA computes whole output tiles) and stream-K (the
 * tiles' 64-wide k-blocks are shared out evenly over one CTA per SM; a tile
 * split across CTAs is summed by the last of them in k order).
 * TRACK_GEMM_DATA_PARALLEL always uses whole tiles; TRACK_GEMM_STREAM_K uses
 * stream-K wherever the shape allows it (every CTA gets at least one k-block
 * and no tile spans more than 4 CTAs), else decides as AUTO.  Every schedule
 * is deterministic (same inputs, same launch: same bits); two schedules differ
 * in fp32 rounding only.  EINVAL for any other mode. */
#define TRACK_GEMM_AUTO 0
#define TRACK_GEMM_DATA_PARALLEL 1
#define TRACK_GEMM_STREAM_K 2
int track_gemm_schedule(int mode);

/* Tile order of the TRACK_BF16 GEMM (process-wide): output tiles are taken in
 * groups of `group` 128-row units, the row unit
 * varying fastest inside a group, then the 128-to-256-column tile.  The tiles
 * running at one time then share few A and W blocks, which stay in L2 while
 * they are reused.  A group at least as large as the row-unit count is plain
 * column order.  0 restores the default, groups of 32.  Data-parallel results do not depend
 * on the order; under stream-K it moves the split points between tiles (fp32
 * rounding only).  EINVAL outside 0..65536. */
int track_gemm_raster(int group);

/* Schedule of the TRACK_BF16 attention kernel (process-wide), with the mode
 * values of track_gemm_schedule, optionally or-ed with
 * TRACK_ATTN_ONE_TILE.  The kernel is persistent, at most one CTA per SM, and
 * its work item is a pair of 128-query tiles of one (sequence, head) sharing
 * every K and V tile it loads; with TRACK_ATTN_ONE_TILE it is the earlier
 * kernel whose item is a single 128-query tile.  TRACK_GEMM_DATA_PARALLEL
 * gives each CTA whole items; TRACK_GEMM_STREAM_K shares the items' 128-key
 * blocks out evenly over one CTA per SM.  It is used wherever no item would
 * span more than 4 CTAs.  A split item is finished by the last of its CTAs,
 * which combines the parts' row maxima, row sums and unnormalized outputs in
 * key order.  TRACK_GEMM_AUTO (the default) picks per launch by a makespan
 * model.  Without TRACK_ATTN_ONE_TILE the one-tile kernel is still taken for
 * key ranges of at most 4 tiles (512 keys) when the pair kernel would have at
 * most two items per SM.  Each schedule is deterministic; they differ in fp32
 * rounding only.  EINVAL for any other mode. */
#define TRACK_ATTN_ONE_TILE 4
int track_attention_schedule(int mode);

/* O = softmax(Q K^T / sqrt(hd)) V per (sequence, head), no mask.  Q: [S, H, Lq,
 * hd], K, V: [S, H, Lk, hd], O: [S, Lq, H, hd], all in dtype (bf16 or fp32);
 * hd in {64, 128}. */
int track_attention(int dtype, const void* Q, const void* K, const void* V, int S, int H,
                    int Lq, int Lk, int hd, void* O, track_stream s);

/* ---- allocation-free variant of track_disagreement -------------------------
 * The paper has no counterpart to this entry point.  It is for callers that
 * cannot allocate device memory while they run: a process whose device memory
 * is reserved up front by its own pool allocator (a cudaMalloc in mid-run could
 * fail), or a latency-critical loop that cannot take the device-wide
 * synchronization that cudaMalloc/cudaFree imply.
 *
 * Computes the relative disagreement score computed by track_disagreement
 * (added to score_accum[b]), with the same arguments, but allocates nothing: its partial
 * sums live in one fixed device array of TRACK_STATIC_MAX_SAMPLES x
 * TRACK_STATIC_MAX_BLOCKS x 2 floats (256 KiB) compiled into the library, which
 * every GPU that loads the library holds until the process exits.
 *  - B above TRACK_STATIC_MAX_SAMPLES is rejected with TRACK_EINVAL.
 *  - s must be a stream of the current device (or NULL): TRACK_EINVAL if not.
 *  - The first call on each device looks up the array's device address
 *    (cudaGetSymbolAddress) with that device current; make that first call
 *    before any stream capture.
 *  - Every call shares the one array: calls whose kernels overlap on the GPU
 *    (two streams with no ordering between them, two host threads) race and
 *    produce wrong scores.  Calls ordered on one stream are safe; each call
 *    writes every scratch slot it reads, so nothing is cleared in between.
 */
#define TRACK_STATIC_MAX_SAMPLES 64
#define TRACK_STATIC_MAX_BLOCKS 512
int track_disagreement_static(const float* v_L, const float* v_S, int B, int64_t n_per_sample,
                              float eps, float* score_accum, track_stream s);

#ifdef __cplusplus
}
#endif

#endif /* TRACK_H */
