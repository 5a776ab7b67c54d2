// Host runtime and C ABI of libtrack: model objects (weights resident in HBM),
// workspaces, the denoiser forward as a sequence of kernel launches on one
// stream, guidance and scheduler calls, the calibration and routed-sampling
// loops of TRACK, and the host-side policy.
#include <cuda_runtime.h>
#include <math.h>
#include <stdio.h>
#include <string.h>

#include <algorithm>
#include <atomic>
#include <map>
#include <unordered_set>
#include <mutex>
#include <string>
#include <utility>
#include <vector>

#include "../../include/track.h"
#include "internal.h"

namespace track {

// ---------------------------------------------------------------- errors and counters
static thread_local std::string g_last_error;

static int fail(int code, const std::string& msg) {
  g_last_error = msg;
  return code;
}

int report_error(int code, const char* msg) { return fail(code, msg); }

#define TRACK_CUDA(expr)                                                              \
  do {                                                                                \
    cudaError_t e_ = (expr);                                                          \
    if (e_ != cudaSuccess)                                                            \
      return fail(TRACK_ECUDA, std::string(#expr) + ": " + cudaGetErrorString(e_));   \
  } while (0)

#define TRACK_TRY(expr)           \
  do {                            \
    int st_ = (expr);             \
    if (st_ != TRACK_OK) return st_; \
  } while (0)

static std::atomic<int64_t> g_launches{0};
void count_launch(int n) { g_launches.fetch_add(n, std::memory_order_relaxed); }

static std::mutex g_dev_mu;
static std::map<int, int> g_sms;
static std::map<int, int*> g_err_words;

static int current_device() {
  int d = 0;
  cudaGetDevice(&d);
  return d;
}

int num_sms() {
  const int dev = current_device();
  std::lock_guard<std::mutex> lk(g_dev_mu);
  auto it = g_sms.find(dev);
  if (it != g_sms.end()) return it->second;
  int n = 0;
  if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || n <= 0) n = 1;
  g_sms[dev] = n;
  return n;
}

// Pending injected allocation failures (track_fail_next_allocations).
static std::atomic<int> g_failing_allocs{0};

void set_failing_allocations(int n) { g_failing_allocs.store(n); }

cudaError_t dev_malloc(void** p, size_t bytes) {
  int pending = g_failing_allocs.load();
  while (pending > 0) {
    if (g_failing_allocs.compare_exchange_weak(pending, pending - 1)) {
      *p = nullptr;
      return cudaErrorMemoryAllocation;
    }
  }
  return cudaMalloc(p, bytes);
}

int* device_error_word() {
  const int dev = current_device();
  std::lock_guard<std::mutex> lk(g_dev_mu);
  auto it = g_err_words.find(dev);
  if (it != g_err_words.end()) return it->second;
  int* p = nullptr;
  if (cudaMalloc(&p, sizeof(int)) != cudaSuccess) return nullptr;
  if (cudaMemset(p, 0, sizeof(int)) != cudaSuccess) return nullptr;
  g_err_words[dev] = p;
  return p;
}

// ---------------------------------------------------------------- profiling
// Timed classes (track_profile_read): work is FLOPs for GEMM and attention,
// algorithmic bytes for the others.
enum ProfClass {
  PROF_GEMM = 0,
  PROF_ATTN = 1,    // self-attention
  PROF_LN = 2,      // LayerNorm-modulate (and the cross-attention LayerNorm)
  PROF_NORM = 3,    // RMSNorm of q/k with 3-D RoPE, in place
  PROF_UPDATE = 4,  // guidance combine and scheduler updates (Eq. 1, Eq. 2)
  PROF_DIS = 5,     // Eq. 4 reduction
  PROF_XATTN = 6,   // cross-attention to the text tokens
  PROF_NCLASS = TRACK_PROFILE_CLASSES
};
struct ProfRec {
  cudaEvent_t a, b;
  int cls;
  double flops;
  bool owned_by_graph = false;  // recorded by a graph's event nodes; never pooled
};
static std::mutex g_prof_mu;
static std::atomic<bool> g_prof_on{false};
static std::vector<ProfRec> g_prof;
static std::vector<std::pair<cudaEvent_t, cudaEvent_t>> g_prof_pool;

// True on a thread while it records a CUDA graph.  With profiling on, the
// brackets of a recorded launch become event-record nodes of the graph; their
// events belong to the graph and are collected in g_capture_recs.
static thread_local bool g_capturing = false;
static thread_local std::vector<ProfRec>* g_capture_recs = nullptr;

struct ProfScope {
  bool on = false;
  ProfRec r;
  cudaStream_t s;
  ProfScope(int cls, double flops, cudaStream_t st) : s(st) {
    if (!g_prof_on.load(std::memory_order_relaxed)) return;
    r.cls = cls;
    r.flops = flops;
    if (g_capturing) {
      if (g_capture_recs == nullptr) return;
      if (cudaEventCreate(&r.a) != cudaSuccess) return;
      if (cudaEventCreate(&r.b) != cudaSuccess) {
        cudaEventDestroy(r.a);
        return;
      }
      r.owned_by_graph = true;
      on = cudaEventRecordWithFlags(r.a, s, cudaEventRecordExternal) == cudaSuccess;
      if (!on) {
        cudaEventDestroy(r.a);
        cudaEventDestroy(r.b);
      }
      return;
    }
    std::lock_guard<std::mutex> lk(g_prof_mu);
    if (!g_prof_pool.empty()) {
      r.a = g_prof_pool.back().first;
      r.b = g_prof_pool.back().second;
      g_prof_pool.pop_back();
    } else {
      if (cudaEventCreate(&r.a) != cudaSuccess) return;
      if (cudaEventCreate(&r.b) != cudaSuccess) return;
    }
    on = cudaEventRecord(r.a, s) == cudaSuccess;
  }
  ~ProfScope() {
    if (!on) return;
    if (r.owned_by_graph) {
      cudaEventRecordWithFlags(r.b, s, cudaEventRecordExternal);
      g_capture_recs->push_back(r);
      return;
    }
    cudaEventRecord(r.b, s);
    std::lock_guard<std::mutex> lk(g_prof_mu);
    g_prof.push_back(r);
  }
};

// ---------------------------------------------------------------- canonical tensors
static const char* kGlobal[12] = {"pe.W", "pe.b", "txt.W1", "txt.b1", "txt.W2", "txt.b2",
                                  "tim.W1", "tim.b1", "tim.W2", "tim.b2", "mod.W", "mod.b"};
static const char* kBlock[27] = {"mod_bias", "q.W",   "q.b",   "k.W",   "k.b",    "v.W",
                                 "v.b",      "o.W",   "o.b",   "qn.g",  "kn.g",   "ln3.g",
                                 "ln3.b",    "cq.W",  "cq.b",  "ck.W",  "ck.b",   "cv.W",
                                 "cv.b",     "co.W",  "co.b",  "cqn.g", "ckn.g",  "ffn.W1",
                                 "ffn.b1",   "ffn.W2", "ffn.b2"};
static const char* kHead[3] = {"head_bias", "head.W", "head.b"};

struct TensorInfo {
  std::string name;  // base name (without block prefix)
  int layer;         // -1 for global / head
  int64_t rows, cols;
  bool matrix;
  char kind;         // 'W' matrix, 'b' bias, 'g' gain (1 + N), 'z' LayerNorm offset
};

static int n_tensors(const track_arch& a) { return 12 + 27 * a.layers + 3; }

static TensorInfo tensor_info(const track_arch& a, int idx) {
  TensorInfo t;
  const int64_t d = a.dim, F = a.ffn, P = (int64_t)a.in_ch * a.patch_f * a.patch_h * a.patch_w;
  if (idx < 12) {
    t.name = kGlobal[idx];
    t.layer = -1;
  } else if (idx < 12 + 27 * a.layers) {
    t.name = kBlock[(idx - 12) % 27];
    t.layer = (idx - 12) / 27;
  } else {
    t.name = kHead[idx - 12 - 27 * a.layers];
    t.layer = -1;
  }
  const std::string& n = t.name;
  t.matrix = n.size() >= 2 && (n.compare(n.size() - 2, 2, ".W") == 0 ||
                               n.compare(n.size() - 3, 3, ".W1") == 0 ||
                               n.compare(n.size() - 3, 3, ".W2") == 0);
  t.cols = 1;
  if (n == "pe.W") { t.rows = d; t.cols = P; }
  else if (n == "txt.W1") { t.rows = d; t.cols = a.text_dim; }
  else if (n == "tim.W1") { t.rows = d; t.cols = a.freq_dim; }
  else if (n == "mod.W") { t.rows = 6 * d; t.cols = d; }
  else if (n == "mod.b") { t.rows = 6 * d; }
  else if (n == "mod_bias") { t.rows = 6; t.cols = d; }
  else if (n == "head_bias") { t.rows = 2; t.cols = d; }
  else if (n == "head.W") { t.rows = P; t.cols = d; }
  else if (n == "head.b") { t.rows = P; }
  else if (n == "ffn.W1") { t.rows = F; t.cols = d; }
  else if (n == "ffn.b1") { t.rows = F; }
  else if (n == "ffn.W2") { t.rows = d; t.cols = F; }
  else if (t.matrix) { t.rows = d; t.cols = d; }
  else { t.rows = d; }
  if (t.matrix) t.kind = 'W';
  else if (n == "qn.g" || n == "kn.g" || n == "cqn.g" || n == "ckn.g" || n == "ln3.g") t.kind = 'g';
  else if (n == "ln3.b") t.kind = 'z';
  else t.kind = 'b';
  return t;
}

// ---------------------------------------------------------------- model object
struct Layer {
  void *Wqkv, *Wo, *Wcq, *Wckv, *Wco, *W1, *W2;
  float *bqkv, *bo, *qn_g, *kn_g, *ln3_g, *ln3_b, *bcq, *bckv, *bco, *cqn_g, *ckn_g, *b1, *b2;
};

struct Workspace {
  int cap = 0;  // capacity in sequences
  void* base = nullptr;
  float* xres = nullptr;
  void *h = nullptr, *qkv = nullptr;
  void *attn = nullptr, *ffh = nullptr;
  float* fout = nullptr;
  // projected text and every block's cross-attention K|V, token-major [Mt, layers * 2d]
  void *ctx_in = nullptr, *ctx_h = nullptr, *ctx_c = nullptr, *ckv = nullptr;
  float *emb = nullptr, *e_tmp = nullptr, *e = nullptr, *e0 = nullptr, *mod_all = nullptr,
        *head_mod = nullptr;
  // guided predictions of calibration (B samples each)
  int calib_cap = 0;
  float *pL = nullptr, *pS = nullptr;
};

}  // namespace track

struct track_model {
  track_arch a;
  int dev = 0;
  int dtype = track::F32;
  size_t esz = 4;
  int L_tok = 0, Fp = 0, Hp = 0, Wp = 0, hd = 0;
  int64_t latent_n = 0;
  void* wbuf = nullptr;
  std::vector<void*> tensor_ptr;  // device destination of each canonical tensor
  void *pe_W, *txt_W1, *txt_W2, *tim_W1, *tim_W2, *mod_W, *head_W;
  float *pe_b, *txt_b1, *txt_b2, *tim_b1, *tim_b2, *mod_b, *mod_bias, *head_bias, *head_b;
  // every block's cross-attention K/V projection, stacked: [layers * 2d, d], [layers * 2d];
  // and the cross-attention key RMSNorm gains [layers, d]
  void* Wckv_all;
  float *bckv_all, *ckn_all;
  std::vector<track::Layer> layer;
  float2* rope_tab = nullptr;
  track::Workspace ws;
  // cache of the projected text conditioning and cross-attention keys/values
  const float* c_cond = nullptr;
  const float* c_uncond = nullptr;
  int c_nseq = -1;
  bool c_valid = false;
  uint64_t ws_gen = 0;  // bumped whenever the workspace is reallocated (graphs hold its addresses)
};

namespace track {

static int validate_arch(const track_arch* a) {
  if (a == nullptr) return fail(TRACK_EINVAL, "arch is NULL");
  if (a->dim <= 0 || a->layers <= 0 || a->heads <= 0 || a->ffn <= 0 || a->text_dim <= 0 ||
      a->text_len <= 0 || a->frames <= 0 || a->height <= 0 || a->width <= 0)
    return fail(TRACK_EINVAL, "arch sizes must be positive");
  if (a->dim % a->heads) return fail(TRACK_EINVAL, "dim must be a multiple of heads");
  const int hd = a->dim / a->heads;
  if (hd != 64 && hd != 128) return fail(TRACK_EINVAL, "head_dim must be 64 or 128");
  if (a->in_ch != 16) return fail(TRACK_EINVAL, "in_ch must be 16");
  if (a->patch_f != 1 || a->patch_h != 2 || a->patch_w != 2)
    return fail(TRACK_EINVAL, "patch must be 1x2x2");
  if (a->height % 2 || a->width % 2) return fail(TRACK_EINVAL, "height and width must be even");
  if (a->freq_dim != 256) return fail(TRACK_EINVAL, "freq_dim must be 256");
  if (a->dim % 64 || a->ffn % 64 || a->text_dim % 64)
    return fail(TRACK_EINVAL, "dim, ffn and text_dim must be multiples of 64");
  if (a->dim > 6144) return fail(TRACK_EINVAL, "dim above 6144 is not supported");
  if (a->dtype != TRACK_FP32 && a->dtype != TRACK_BF16) return fail(TRACK_EINVAL, "bad dtype");
  if (!(a->eps > 0.f)) return fail(TRACK_EINVAL, "eps must be positive");
  return TRACK_OK;
}

static void* dalloc_carve(uint8_t*& p, size_t bytes) {
  void* r = p;
  p += (bytes + 255) & ~(size_t)255;
  return r;
}

// Lays out all weights in one allocation; fills the model's pointers and the
// destination of every canonical tensor.  With base == nullptr only sizes.
static size_t layout_weights(track_model* m, uint8_t* base) {
  const track_arch& a = m->a;
  const int64_t d = a.dim, F = a.ffn, Dt = a.text_dim, P = 64;
  const size_t es = m->esz;
  uint8_t* p = base;
  auto mat = [&](int64_t r, int64_t c) { return dalloc_carve(p, (size_t)(r * c) * es); };
  auto vec = [&](int64_t n) { return (float*)dalloc_carve(p, (size_t)n * 4); };
  m->pe_W = mat(d, P); m->pe_b = vec(d);
  m->txt_W1 = mat(d, Dt); m->txt_b1 = vec(d); m->txt_W2 = mat(d, d); m->txt_b2 = vec(d);
  m->tim_W1 = mat(d, a.freq_dim); m->tim_b1 = vec(d); m->tim_W2 = mat(d, d); m->tim_b2 = vec(d);
  m->mod_W = mat(6 * d, d); m->mod_b = vec(6 * d);
  m->mod_bias = vec((int64_t)a.layers * 6 * d);
  m->Wckv_all = mat((int64_t)a.layers * 2 * d, d);
  m->bckv_all = vec((int64_t)a.layers * 2 * d);
  m->ckn_all = vec((int64_t)a.layers * d);
  m->layer.resize(a.layers);
  for (int l = 0; l < a.layers; ++l) {
    Layer& L = m->layer[l];
    L.Wqkv = mat(3 * d, d); L.bqkv = vec(3 * d);
    L.Wo = mat(d, d); L.bo = vec(d);
    L.qn_g = vec(d); L.kn_g = vec(d); L.ln3_g = vec(d); L.ln3_b = vec(d);
    L.Wcq = mat(d, d); L.bcq = vec(d);
    L.Wckv = (uint8_t*)m->Wckv_all + (size_t)l * 2 * d * d * es;
    L.bckv = m->bckv_all + (int64_t)l * 2 * d;
    L.Wco = mat(d, d); L.bco = vec(d);
    L.cqn_g = vec(d); L.ckn_g = m->ckn_all + (int64_t)l * d;
    L.W1 = mat(F, d); L.b1 = vec(F);
    L.W2 = mat(d, F); L.b2 = vec(d);
  }
  m->head_bias = vec(2 * d); m->head_W = mat(P, d); m->head_b = vec(P);
  const size_t total = (size_t)(p - base);
  if (base == nullptr) return total;

  const int nt = n_tensors(a);
  m->tensor_ptr.assign(nt, nullptr);
  for (int i = 0; i < nt; ++i) {
    const TensorInfo t = tensor_info(a, i);
    const std::string& n = t.name;
    uint8_t* dst = nullptr;
    if (t.layer < 0) {
      if (n == "pe.W") dst = (uint8_t*)m->pe_W;
      else if (n == "pe.b") dst = (uint8_t*)m->pe_b;
      else if (n == "txt.W1") dst = (uint8_t*)m->txt_W1;
      else if (n == "txt.b1") dst = (uint8_t*)m->txt_b1;
      else if (n == "txt.W2") dst = (uint8_t*)m->txt_W2;
      else if (n == "txt.b2") dst = (uint8_t*)m->txt_b2;
      else if (n == "tim.W1") dst = (uint8_t*)m->tim_W1;
      else if (n == "tim.b1") dst = (uint8_t*)m->tim_b1;
      else if (n == "tim.W2") dst = (uint8_t*)m->tim_W2;
      else if (n == "tim.b2") dst = (uint8_t*)m->tim_b2;
      else if (n == "mod.W") dst = (uint8_t*)m->mod_W;
      else if (n == "mod.b") dst = (uint8_t*)m->mod_b;
      else if (n == "head_bias") dst = (uint8_t*)m->head_bias;
      else if (n == "head.W") dst = (uint8_t*)m->head_W;
      else if (n == "head.b") dst = (uint8_t*)m->head_b;
    } else {
      Layer& L = m->layer[t.layer];
      const size_t md = (size_t)(d * d) * es;  // one [d, d] matrix
      if (n == "mod_bias") dst = (uint8_t*)(m->mod_bias + (int64_t)t.layer * 6 * d);
      else if (n == "q.W") dst = (uint8_t*)L.Wqkv;
      else if (n == "k.W") dst = (uint8_t*)L.Wqkv + md;
      else if (n == "v.W") dst = (uint8_t*)L.Wqkv + 2 * md;
      else if (n == "q.b") dst = (uint8_t*)L.bqkv;
      else if (n == "k.b") dst = (uint8_t*)(L.bqkv + d);
      else if (n == "v.b") dst = (uint8_t*)(L.bqkv + 2 * d);
      else if (n == "o.W") dst = (uint8_t*)L.Wo;
      else if (n == "o.b") dst = (uint8_t*)L.bo;
      else if (n == "qn.g") dst = (uint8_t*)L.qn_g;
      else if (n == "kn.g") dst = (uint8_t*)L.kn_g;
      else if (n == "ln3.g") dst = (uint8_t*)L.ln3_g;
      else if (n == "ln3.b") dst = (uint8_t*)L.ln3_b;
      else if (n == "cq.W") dst = (uint8_t*)L.Wcq;
      else if (n == "cq.b") dst = (uint8_t*)L.bcq;
      else if (n == "ck.W") dst = (uint8_t*)L.Wckv;
      else if (n == "cv.W") dst = (uint8_t*)L.Wckv + md;
      else if (n == "ck.b") dst = (uint8_t*)L.bckv;
      else if (n == "cv.b") dst = (uint8_t*)(L.bckv + d);
      else if (n == "co.W") dst = (uint8_t*)L.Wco;
      else if (n == "co.b") dst = (uint8_t*)L.bco;
      else if (n == "cqn.g") dst = (uint8_t*)L.cqn_g;
      else if (n == "ckn.g") dst = (uint8_t*)L.ckn_g;
      else if (n == "ffn.W1") dst = (uint8_t*)L.W1;
      else if (n == "ffn.b1") dst = (uint8_t*)L.b1;
      else if (n == "ffn.W2") dst = (uint8_t*)L.W2;
      else if (n == "ffn.b2") dst = (uint8_t*)L.b2;
    }
    m->tensor_ptr[i] = dst;
  }
  return total;
}

static int build_rope_table(track_model* m) {
  const int hd = m->hd, s6 = hd / 6;
  const int df = hd - 4 * s6, dh = 2 * s6;
  const int nf = df / 2, nh = s6;
  std::vector<float2> tab((size_t)m->Fp * nf + (size_t)m->Hp * nh + (size_t)m->Wp * nh);
  size_t o = 0;
  for (int p = 0; p < m->Fp; ++p)
    for (int j = 0; j < nf; ++j) {
      const double ang = p * pow(10000.0, -2.0 * j / df);
      tab[o++] = make_float2((float)cos(ang), (float)sin(ang));
    }
  for (int ax = 0; ax < 2; ++ax) {
    const int n = ax == 0 ? m->Hp : m->Wp;
    for (int p = 0; p < n; ++p)
      for (int j = 0; j < nh; ++j) {
        const double ang = p * pow(10000.0, -2.0 * j / dh);
        tab[o++] = make_float2((float)cos(ang), (float)sin(ang));
      }
  }
  if (dev_malloc((void**)&m->rope_tab, tab.size() * sizeof(float2)) != cudaSuccess) {
    cudaGetLastError();
    m->rope_tab = nullptr;
    return fail(TRACK_ENOMEM, "rope table allocation failed");
  }
  TRACK_CUDA(cudaMemcpy(m->rope_tab, tab.data(), tab.size() * sizeof(float2),
                        cudaMemcpyHostToDevice));
  return TRACK_OK;
}

static void free_workspace(Workspace& w) {
  if (w.base) cudaFree(w.base);
  if (w.pL) cudaFree(w.pL);
  w = Workspace();
}

static int ensure_workspace(track_model* m, int nseq) {
  Workspace& w = m->ws;
  if (nseq <= w.cap) return TRACK_OK;
  const int calib_cap = w.calib_cap;
  float* pL = w.pL;
  float* pS = w.pS;
  if (w.base) cudaFree(w.base);
  w.base = nullptr;
  w.cap = 0;
  m->c_valid = false;
  ++m->ws_gen;
  const track_arch& a = m->a;
  const int64_t d = a.dim, F = a.ffn, Lt = a.text_len, Dt = a.text_dim;
  const int64_t M = (int64_t)nseq * m->L_tok, Mt = (int64_t)nseq * Lt;
  const size_t es = m->esz;
  size_t need = 0;
  auto sz = [&](size_t b) { need += (b + 255) & ~(size_t)255; };
  sz(M * d * 4);                       // xres
  sz(M * d * es);                      // h
  sz(M * 3 * d * es);                  // qkv
  sz(M * d * es);                      // attn
  sz(M * F * es);                      // ffh
  sz((size_t)nseq * m->latent_n * 4);  // fout
  sz(Mt * Dt * es);                    // ctx_in
  sz(Mt * d * es);                     // ctx_h
  sz(Mt * d * es);                     // ctx_c
  sz((size_t)Mt * a.layers * 2 * d * es);  // ckv (all blocks)
  sz(256 * 4);
  sz(d * 4);
  sz(d * 4);
  sz(6 * d * 4);
  sz((size_t)a.layers * 6 * d * 4);
  sz(2 * d * 4);
  void* base = nullptr;
  cudaError_t e = dev_malloc((void**)&base, need);
  if (e != cudaSuccess) {
    cudaGetLastError();
    return fail(TRACK_ENOMEM, std::string("workspace allocation failed: ") + cudaGetErrorString(e));
  }
  uint8_t* p = (uint8_t*)base;
  w.base = base;
  w.xres = (float*)dalloc_carve(p, M * d * 4);
  w.h = dalloc_carve(p, M * d * es);
  w.qkv = dalloc_carve(p, M * 3 * d * es);
  w.attn = dalloc_carve(p, M * d * es);
  w.ffh = dalloc_carve(p, M * F * es);
  w.fout = (float*)dalloc_carve(p, (size_t)nseq * m->latent_n * 4);
  w.ctx_in = dalloc_carve(p, Mt * Dt * es);
  w.ctx_h = dalloc_carve(p, Mt * d * es);
  w.ctx_c = dalloc_carve(p, Mt * d * es);
  w.ckv = dalloc_carve(p, (size_t)Mt * a.layers * 2 * d * es);
  w.emb = (float*)dalloc_carve(p, 256 * 4);
  w.e_tmp = (float*)dalloc_carve(p, d * 4);
  w.e = (float*)dalloc_carve(p, d * 4);
  w.e0 = (float*)dalloc_carve(p, 6 * d * 4);
  w.mod_all = (float*)dalloc_carve(p, (size_t)a.layers * 6 * d * 4);
  w.head_mod = (float*)dalloc_carve(p, 2 * d * 4);
  w.cap = nseq;
  w.calib_cap = calib_cap;
  w.pL = pL;
  w.pS = pS;
  return TRACK_OK;
}

static int ensure_calib(track_model* m, int B) {
  Workspace& w = m->ws;
  if (B <= w.calib_cap) return TRACK_OK;
  if (w.pL) cudaFree(w.pL);
  w.pL = w.pS = nullptr;
  w.calib_cap = 0;
  const size_t n = (size_t)B * m->latent_n;
  float* p = nullptr;
  if (dev_malloc((void**)&p, 2 * n * sizeof(float)) != cudaSuccess) {
    cudaGetLastError();
    return fail(TRACK_ENOMEM, "calibration buffers");
  }
  w.pL = p;
  w.pS = p + n;
  w.calib_cap = B;
  return TRACK_OK;
}

// ---------------------------------------------------------------- GEMM / attention dispatch
static int run_gemm(const track_model* m, const void* A, const void* W, int M, int N, int K,
                    const float* bias, int epi, const float* gate, void* out, int ldo,
                    cudaStream_t s) {
  GemmArgs g;
  g.M = M; g.N = N; g.K = K; g.epi = epi; g.bias = bias; g.gate = gate; g.out = out; g.ldo = ldo;
  g.w_static = 1;  // W is a weight of the model
  g.err = device_error_word();
  if (g.err == nullptr) return fail(TRACK_ECUDA, "device error word allocation failed");
  ProfScope ps(PROF_GEMM, 2.0 * M * N * (double)K, s);
  cudaError_t e = m->dtype == BF16 ? gemm_bf16_tc(A, W, g, s)
                                   : gemm_f32((const float*)A, (const float*)W, g, s);
  if (e != cudaSuccess)
    return fail(TRACK_ECUDA, std::string("gemm launch: ") + cudaGetErrorString(e));
  return TRACK_OK;
}

static int run_attention(const track_model* m, const AttnOperand& Q, const AttnOperand& K,
                         const AttnOperand& V, void* O, int S, int Lq, int Lk, cudaStream_t s) {
  const int H = m->a.heads, hd = m->hd;
  ProfScope ps(Lq == Lk ? PROF_ATTN : PROF_XATTN, 4.0 * S * H * (double)Lq * Lk * hd, s);
  cudaError_t e = m->dtype == BF16 ? attention_bf16(Q, K, V, O, S, H, Lq, Lk, hd, s)
                                   : attention_f32(Q, K, V, (float*)O, S, H, Lq, Lk, hd, s);
  if (e != cudaSuccess)
    return fail(TRACK_ECUDA, std::string("attention launch: ") + cudaGetErrorString(e));
  return TRACK_OK;
}

// LayerNorm-modulate (class 2) and in-place RMSNorm/RoPE (class 3) launches,
// timed with their algorithmic bytes (fp32 row in + activation row out;
// activation in + out).
static cudaError_t run_ln(const track_model* m, const float* x, int M, int d, const float* a,
                          const float* b, int mode, void* out, cudaStream_t s) {
  ProfScope ps(PROF_LN, (double)M * d * (4.0 + m->esz), s);
  return ln_modulate(x, M, d, a, b, mode, m->a.eps, out, m->dtype, s);
}
static cudaError_t run_norm(const track_model* m, const NormRopeArgs& p, cudaStream_t s) {
  ProfScope ps(PROF_NORM, (double)p.rows * p.d * p.nsec * 2.0 * m->esz, s);
  return qk_norm_rope(p, s);
}

static NormRopeArgs norm_args(const track_model* m, void* buf, int ld, int rows, int L) {
  NormRopeArgs p;
  memset(&p, 0, sizeof(p));
  p.buf = buf; p.ld = ld; p.rows = rows; p.L = L; p.hd = m->hd; p.d = m->a.dim;
  p.rope_tab = m->rope_tab; p.Fp = m->Fp; p.Hp = m->Hp; p.Wp = m->Wp;
  p.eps = m->a.eps; p.dtype = m->dtype;
  return p;
}

#define LAUNCH(expr)                                                                  \
  do {                                                                                \
    cudaError_t e_ = (expr);                                                          \
    if (e_ != cudaSuccess)                                                            \
      return fail(TRACK_ECUDA, std::string(#expr) + ": " + cudaGetErrorString(e_));   \
  } while (0)

// Text projection and per-block cross-attention keys/values for nseq sequences.
static int project_context(track_model* m, const float* cond, const float* uncond, int B,
                           int nseq, cudaStream_t s) {
  if (m->c_valid && m->c_cond == cond && m->c_uncond == uncond && m->c_nseq == nseq)
    return TRACK_OK;
  const track_arch& a = m->a;
  Workspace& w = m->ws;
  const int64_t d = a.dim, Lt = a.text_len, Dt = a.text_dim;
  const int Mt = nseq * (int)Lt;
  const int64_t per = (int64_t)B * Lt * Dt;
  LAUNCH(convert_f32(cond, w.ctx_in, m->dtype, per, s));
  if (nseq > B) LAUNCH(convert_f32(uncond, (uint8_t*)w.ctx_in + per * m->esz, m->dtype, per, s));
  TRACK_TRY(run_gemm(m, w.ctx_in, m->txt_W1, Mt, (int)d, (int)Dt, m->txt_b1, EPI_GELU, nullptr,
                     w.ctx_h, (int)d, s));
  TRACK_TRY(run_gemm(m, w.ctx_h, m->txt_W2, Mt, (int)d, (int)d, m->txt_b2, EPI_STORE, nullptr,
                     w.ctx_c, (int)d, s));
  // every block's cross-attention K|V in one GEMM, then RMSNorm of every block's K in place
  const int nkv = a.layers * 2 * (int)d;
  TRACK_TRY(run_gemm(m, w.ctx_c, m->Wckv_all, Mt, nkv, (int)d, m->bckv_all, EPI_STORE, nullptr,
                     w.ckv, nkv, s));
  NormRopeArgs p = norm_args(m, w.ckv, nkv, Mt, (int)Lt);
  p.nsec = a.layers; p.off0 = 0; p.off_stride = 2 * d;
  p.gain0 = m->ckn_all; p.gain_stride = d;
  p.rope = 0;
  LAUNCH(run_norm(m, p, s));
  m->c_cond = cond;
  m->c_uncond = uncond;
  m->c_nseq = nseq;
  m->c_valid = true;
  return TRACK_OK;
}

// f_m(x, t, c) for nseq = B (cond) or 2B (cond then uncond) sequences -> out [nseq, C, F, H, W].
static int forward(track_model* m, const float* x, int B, int nseq, float t, const float* cond,
                   const float* uncond, float* out, cudaStream_t s) {
  const track_arch& a = m->a;
  TRACK_TRY(ensure_workspace(m, nseq));
  Workspace& w = m->ws;
  const int d = a.dim, F = a.ffn, L = m->L_tok;
  const int M = nseq * L;
  const size_t es = m->esz;

  // timestep embedding and modulation vectors (shared by all sequences)
  LAUNCH(sinusoid(t, w.emb, a.freq_dim, s));
  LAUNCH(matvec(m->tim_W1, m->dtype, w.emb, m->tim_b1, w.e_tmp, d, a.freq_dim, 0, s));
  LAUNCH(matvec(m->tim_W2, m->dtype, w.e_tmp, m->tim_b2, w.e, d, d, 1, s));
  LAUNCH(matvec(m->mod_W, m->dtype, w.e, m->mod_b, w.e0, 6 * d, d, 1, s));
  LAUNCH(modulation(w.e0, m->mod_bias, a.layers, w.e, m->head_bias, d, w.mod_all, w.head_mod, s));

  TRACK_TRY(project_context(m, cond, uncond, B, nseq, s));
  LAUNCH(patch_embed(x, B, nseq, a.in_ch, a.frames, a.height, a.width, m->pe_W, m->dtype, m->pe_b,
                     d, w.xres, s));

  const int nkv = a.layers * 2 * d;

  for (int l = 0; l < a.layers; ++l) {
    const Layer& Ly = m->layer[l];
    const float* mod = w.mod_all + (size_t)l * 6 * d;
    const float *shift1 = mod, *scale1 = mod + d, *gate1 = mod + 2 * d;
    const float *shift2 = mod + 3 * d, *scale2 = mod + 4 * d, *gate2 = mod + 5 * d;
    // self-attention
    LAUNCH(run_ln(m, w.xres, M, d, scale1, shift1, 0, w.h, s));
    TRACK_TRY(run_gemm(m, w.h, Ly.Wqkv, M, 3 * d, d, Ly.bqkv, EPI_STORE, nullptr, w.qkv, 3 * d, s));
    {  // q and k: RMSNorm over d and 3D RoPE, in place; v is used as projected
      NormRopeArgs p = norm_args(m, w.qkv, 3 * d, M, L);
      p.nsec = 2; p.off0 = 0; p.off_stride = d;
      p.gain0 = Ly.qn_g; p.gain_stride = Ly.kn_g - Ly.qn_g;
      p.rope = 1;
      LAUNCH(run_norm(m, p, s));
    }
    const uint8_t* qkv = (const uint8_t*)w.qkv;
    TRACK_TRY(run_attention(m, token_major(qkv, L, 3 * d, m->hd),
                            token_major(qkv + (size_t)d * es, L, 3 * d, m->hd),
                            token_major(qkv + (size_t)2 * d * es, L, 3 * d, m->hd), w.attn, nseq, L,
                            L, s));
    TRACK_TRY(run_gemm(m, w.attn, Ly.Wo, M, d, d, Ly.bo, EPI_RESID_GATE, gate1, w.xres, d, s));
    // cross-attention
    LAUNCH(run_ln(m, w.xres, M, d, Ly.ln3_g, Ly.ln3_b, 1, w.h, s));
    TRACK_TRY(run_gemm(m, w.h, Ly.Wcq, M, d, d, Ly.bcq, EPI_STORE, nullptr, w.qkv, d, s));
    {  // cross-attention q: RMSNorm over d, in place
      NormRopeArgs p = norm_args(m, w.qkv, d, M, L);
      p.nsec = 1; p.off0 = 0; p.off_stride = 0;
      p.gain0 = Ly.cqn_g; p.gain_stride = 0;
      p.rope = 0;
      LAUNCH(run_norm(m, p, s));
    }
    const uint8_t* kvl = (const uint8_t*)w.ckv + (size_t)l * 2 * d * es;
    TRACK_TRY(run_attention(m, token_major(w.qkv, L, d, m->hd),
                            token_major(kvl, a.text_len, nkv, m->hd),
                            token_major(kvl + (size_t)d * es, a.text_len, nkv, m->hd), w.attn, nseq,
                            L, a.text_len, s));
    TRACK_TRY(run_gemm(m, w.attn, Ly.Wco, M, d, d, Ly.bco, EPI_RESID, nullptr, w.xres, d, s));
    // MLP
    LAUNCH(run_ln(m, w.xres, M, d, scale2, shift2, 0, w.h, s));
    TRACK_TRY(run_gemm(m, w.h, Ly.W1, M, F, d, Ly.b1, EPI_GELU, nullptr, w.ffh, F, s));
    TRACK_TRY(run_gemm(m, w.ffh, Ly.W2, M, d, F, Ly.b2, EPI_RESID_GATE, gate2, w.xres, d, s));
  }
  // Head: LN(x)(1 + scale) + shift (a11), then its Linear(d -> 4C) as a GEMM into
  // token-major fp32 (the FFN hidden buffer is free after the last block), then
  // unpatchify.
  const int P = 4 * a.in_ch;
  if ((m->dtype == F32 || P % 32 == 0) && (size_t)F * es >= (size_t)P * sizeof(float)) {
    LAUNCH(run_ln(m, w.xres, M, d, w.head_mod + d, w.head_mod, 0, w.h, s));
    float* hv = (float*)w.ffh;
    TRACK_CUDA(cudaMemsetAsync(hv, 0, (size_t)M * P * sizeof(float), s));
    TRACK_TRY(run_gemm(m, w.h, m->head_W, M, P, d, m->head_b, EPI_RESID, nullptr, hv, P, s));
    LAUNCH(unpatchify(hv, nseq, L, a.in_ch, a.frames, a.height, a.width, out, s));
  } else {
    LAUNCH(head_unpatchify(w.xres, nseq, L, d, w.head_mod, m->head_W, m->dtype, m->head_b, a.eps,
                           a.in_ch, a.frames, a.height, a.width, out, s));
  }
  return TRACK_OK;
}

static int check_denoise_args(track_model* m, const void* x, int B, const float* cond,
                              const float* uncond, float w, const void* out) {
  if (m == nullptr) return fail(TRACK_EINVAL, "model is NULL");
  if (x == nullptr || out == nullptr || cond == nullptr) return fail(TRACK_EINVAL, "NULL pointer");
  if (B <= 0) return fail(TRACK_EINVAL, "B must be positive");
  if (!isfinite(w)) return fail(TRACK_EINVAL, "cfg_scale must be finite");
  if (w != 1.f && uncond == nullptr)
    return fail(TRACK_EINVAL, "uncond may be NULL only when cfg_scale == 1");
  if ((((uintptr_t)x) | ((uintptr_t)out) | ((uintptr_t)cond) | ((uintptr_t)uncond)) & 15)
    return fail(TRACK_EINVAL, "device pointers must be 16-byte aligned");
  return TRACK_OK;
}

static int set_device(const track_model* m) {
  int cur = 0;
  TRACK_CUDA(cudaGetDevice(&cur));
  if (cur != m->dev) TRACK_CUDA(cudaSetDevice(m->dev));
  return TRACK_OK;
}

static int denoise_impl(track_model* m, const float* x, int B, float t, const float* cond,
                        const float* uncond, float w, float* v_out, cudaStream_t s) {
  const int nseq = w == 1.f ? B : 2 * B;
  if (w == 1.f) return forward(m, x, B, nseq, t, cond, nullptr, v_out, s);
  TRACK_TRY(ensure_workspace(m, nseq));  // ws.fout is read below: allocate first
  TRACK_TRY(forward(m, x, B, nseq, t, cond, uncond, m->ws.fout, s));
  const int64_t n = (int64_t)B * m->latent_n;
  ProfScope ps(PROF_UPDATE, 12.0 * n, s);  // read f_c, f_u; write p
  LAUNCH(cfg_combine(m->ws.fout, m->ws.fout + n, n, w, v_out, s));
  return TRACK_OK;
}

static int denoise_step_impl(track_model* m, float* x, int B, float sigma_t, float sigma_next,
                             const float* cond, const float* uncond, float w, cudaStream_t s) {
  const int nseq = w == 1.f ? B : 2 * B;
  const float t = 1000.f * sigma_t;
  TRACK_TRY(ensure_workspace(m, nseq));  // ws.fout is read below: allocate first
  TRACK_TRY(forward(m, x, B, nseq, t, cond, w == 1.f ? nullptr : uncond, m->ws.fout, s));
  const int64_t n = (int64_t)B * m->latent_n;
  ProfScope ps(PROF_UPDATE, (w == 1.f ? 12.0 : 16.0) * n, s);  // read f_c (f_u), x; write x
  LAUNCH(cfg_euler(x, m->ws.fout, w == 1.f ? nullptr : m->ws.fout + n, n, w, sigma_next - sigma_t,
                   s));
  return TRACK_OK;
}

// ---------------------------------------------------------------- disagreement scratch
static std::mutex g_scr_mu;
static std::map<std::pair<int, cudaStream_t>, std::pair<float*, size_t>> g_scratch;

static float* stream_scratch(cudaStream_t s, size_t floats) {
  const int dev = current_device();
  std::lock_guard<std::mutex> lk(g_scr_mu);
  auto& slot = g_scratch[std::make_pair(dev, s)];
  if (slot.second >= floats) return slot.first;
  if (slot.first) {
    cudaStreamSynchronize(s);
    cudaFree(slot.first);
  }
  slot.first = nullptr;
  slot.second = 0;
  float* p = nullptr;
  if (dev_malloc((void**)&p, floats * sizeof(float)) != cudaSuccess) {
    cudaGetLastError();
    return nullptr;
  }
  slot.first = p;
  slot.second = floats;
  return p;
}

static int band_impl(const float* vL, const float* vS, int B, int C, int F, int H, int W,
                     float eps, float* out, cudaStream_t s) {
  float* scr = stream_scratch(s, band_scratch_floats(B, C, F, H, W));
  if (scr == nullptr) return fail(TRACK_ENOMEM, "band scratch allocation failed");
  LAUNCH(band_disagreement(vL, vS, B, C, F, H, W, eps, out, scr, s));
  return TRACK_OK;
}

// Per-sample completion counters of the one-launch Eq. 4 reduction, one array
// per (device, stream), zeroed when allocated; every call leaves them at zero.
static std::mutex g_cnt_mu;
static std::map<std::pair<int, cudaStream_t>, std::pair<int*, int>> g_dis_cnt;

static int* dis_counters(cudaStream_t s, int B) {
  const int dev = current_device();
  std::lock_guard<std::mutex> lk(g_cnt_mu);
  auto& slot = g_dis_cnt[std::make_pair(dev, s)];
  if (slot.second >= B) return slot.first;
  if (slot.first) {
    cudaStreamSynchronize(s);
    cudaFree(slot.first);
  }
  slot.first = nullptr;
  slot.second = 0;
  const int n = B > 64 ? B : 64;
  int* p = nullptr;
  if (dev_malloc((void**)&p, n * sizeof(int)) != cudaSuccess ||
      cudaMemsetAsync(p, 0, n * sizeof(int), s) != cudaSuccess) {
    cudaGetLastError();
    cudaFree(p);
    return nullptr;
  }
  slot.first = p;
  slot.second = n;
  return p;
}

// Eq. 4 into accum; with x non-null also x += dsig * vL (Euler, Eq. 2) in the
// same pass.
static int disagreement_impl(const float* vL, const float* vS, int B, int64_t n, float eps,
                             float* accum, cudaStream_t s, float* x = nullptr, float dsig = 0.f) {
  const int nblk = disagreement_blocks(n, B);
  float* scr = stream_scratch(s, (size_t)B * nblk * 2);
  if (scr == nullptr) return fail(TRACK_ENOMEM, "disagreement scratch allocation failed");
  int* cnt = dis_counters(s, B);
  if (cnt == nullptr) return fail(TRACK_ENOMEM, "disagreement counter allocation failed");
  // read p_L, p_S (and x, written back)
  ProfScope ps(PROF_DIS, (x != nullptr ? 16.0 : 8.0) * B * (double)n, s);
  LAUNCH(disagreement_fused(vL, vS, B, n, eps, accum, scr, cnt, nblk, s, x, dsig));
  return TRACK_OK;
}

}  // namespace track

// ====================================================================== C ABI
using namespace track;

// SplitMix64 output mixing (Steele, Lea and Flood 2014), host side.
static uint64_t mix64_host(uint64_t z) {
  z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
  z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
  return z ^ (z >> 31);
}

extern "C" {

const char* track_last_error(void) { return g_last_error.c_str(); }

int track_abi_version(void) { return 1; }

int64_t track_launch_count(void) { return g_launches.load(); }

int track_sync(track_stream s) {
  cudaError_t e = cudaStreamSynchronize((cudaStream_t)s);
  if (e != cudaSuccess) return fail(TRACK_ECUDA, std::string("stream sync: ") + cudaGetErrorString(e));
  int* w = device_error_word();
  if (w == nullptr) return fail(TRACK_ECUDA, "device error word");
  int v = 0;
  TRACK_CUDA(cudaMemcpy(&v, w, sizeof(int), cudaMemcpyDeviceToHost));
  if (v != 0) {
    TRACK_CUDA(cudaMemset(w, 0, sizeof(int)));
    char buf[96];
    snprintf(buf, sizeof(buf), "a kernel abandoned a pipeline wait (code %d)", v);
    return fail(TRACK_ETIMEOUT, buf);
  }
  return TRACK_OK;
}

int track_gemm_schedule(int mode) {
  if (mode < TRACK_GEMM_AUTO || mode > TRACK_GEMM_STREAM_K)
    return fail(TRACK_EINVAL, "unknown GEMM schedule");
  set_gemm_schedule(mode);
  return TRACK_OK;
}

int track_fail_next_allocations(int n) {
  if (n < 0) return fail(TRACK_EINVAL, "n must be non-negative");
  set_failing_allocations(n);
  return TRACK_OK;
}

int track_wait_selftest(int64_t limit_cycles, track_stream s) {
  if (limit_cycles < 1000 || limit_cycles > 2000000000LL)
    return fail(TRACK_EINVAL, "limit_cycles outside 1e3 .. 2e9");
  int* err = device_error_word();
  if (err == nullptr) return fail(TRACK_ECUDA, "device error word");
  cudaError_t e = wait_selftest(err, (long long)limit_cycles, TRACK_WAIT_SELFTEST_CODE, (cudaStream_t)s);
  if (e != cudaSuccess) return fail(TRACK_ECUDA, std::string("self-test launch: ") + cudaGetErrorString(e));
  return TRACK_OK;
}

int track_gemm_raster(int group) {
  if (group < 0 || group > 65536) return fail(TRACK_EINVAL, "raster group out of range");
  set_gemm_raster(group);
  return TRACK_OK;
}

int track_attention_schedule(int mode) {
  if ((mode & ~TRACK_ATTN_ONE_TILE) < TRACK_GEMM_AUTO ||
      (mode & ~TRACK_ATTN_ONE_TILE) > TRACK_GEMM_STREAM_K)
    return fail(TRACK_EINVAL, "unknown attention schedule");
  set_attention_schedule(mode);
  return TRACK_OK;
}

int track_profile_enable(int enable) {
  g_prof_on.store(enable != 0);
  return TRACK_OK;
}

int track_profile_read(double* ms, double* flops, int64_t* launches) {
  if (!ms || !flops || !launches) return fail(TRACK_EINVAL, "NULL output");
  std::lock_guard<std::mutex> lk(g_prof_mu);
  for (int c = 0; c < PROF_NCLASS; ++c) {
    ms[c] = 0;
    flops[c] = 0;
    launches[c] = 0;
  }
  int rc = TRACK_OK;
  for (auto& r : g_prof) {
    float t = 0.f;
    if (cudaEventSynchronize(r.b) != cudaSuccess || cudaEventElapsedTime(&t, r.a, r.b) != cudaSuccess) {
      rc = fail(TRACK_ECUDA, "profile event");
    } else {
      ms[r.cls] += t;
      flops[r.cls] += r.flops;
      launches[r.cls] += 1;
    }
    if (!r.owned_by_graph) g_prof_pool.emplace_back(r.a, r.b);
  }
  g_prof.clear();
  return rc;
}

int track_weight_count(const track_arch* arch) {
  if (validate_arch(arch) != TRACK_OK) return -1;
  return n_tensors(*arch);
}

int track_weight_shape(const track_arch* arch, int index, int64_t* rows, int64_t* cols) {
  TRACK_TRY(validate_arch(arch));
  if (index < 0 || index >= n_tensors(*arch) || !rows || !cols)
    return fail(TRACK_EINVAL, "bad tensor index or NULL output");
  const TensorInfo t = tensor_info(*arch, index);
  *rows = t.rows;
  *cols = t.cols;
  return TRACK_OK;
}

static int model_alloc(const track_arch* arch, track_model** out, track_model** mp) {
  TRACK_TRY(validate_arch(arch));
  if (out == nullptr) return fail(TRACK_EINVAL, "out is NULL");
  *out = nullptr;
  track_model* m = new (std::nothrow) track_model();
  if (!m) return fail(TRACK_ENOMEM, "host allocation");
  m->a = *arch;
  if (cudaGetDevice(&m->dev) != cudaSuccess) {
    delete m;
    return fail(TRACK_ECUDA, "cudaGetDevice");
  }
  m->dtype = arch->dtype == TRACK_BF16 ? BF16 : F32;
  m->esz = m->dtype == BF16 ? 2 : 4;
  m->hd = arch->dim / arch->heads;
  m->Fp = arch->frames;
  m->Hp = arch->height / 2;
  m->Wp = arch->width / 2;
  m->L_tok = m->Fp * m->Hp * m->Wp;
  m->latent_n = (int64_t)arch->in_ch * arch->frames * arch->height * arch->width;
  const size_t bytes = layout_weights(m, nullptr);
  if (dev_malloc((void**)&m->wbuf, bytes) != cudaSuccess) {
    cudaGetLastError();
    delete m;
    return fail(TRACK_ENOMEM, "weight allocation failed");
  }
  layout_weights(m, (uint8_t*)m->wbuf);
  int rc = build_rope_table(m);
  if (rc != TRACK_OK) {
    cudaFree(m->wbuf);
    delete m;
    return rc;
  }
  *mp = m;
  return TRACK_OK;
}

static void drop_graphs_of(const track_model* m);

int track_model_destroy(track_model* m) {
  if (m == nullptr) return TRACK_OK;
  set_device(m);
  cudaDeviceSynchronize();
  drop_graphs_of(m);
  free_workspace(m->ws);
  if (m->wbuf) cudaFree(m->wbuf);
  if (m->rope_tab) cudaFree(m->rope_tab);
  delete m;
  return TRACK_OK;
}

int track_model_create(const track_arch* arch, const float* const* weights, track_model** out) {
  track_model* m = nullptr;
  if (weights == nullptr) return fail(TRACK_EINVAL, "weights is NULL");
  TRACK_TRY(model_alloc(arch, out, &m));
  const int nt = n_tensors(m->a);
  size_t maxn = 0;
  for (int i = 0; i < nt; ++i) {
    if (weights[i] == nullptr) {
      track_model_destroy(m);
      return fail(TRACK_EINVAL, "weights[" + std::to_string(i) + "] is NULL");
    }
    const TensorInfo t = tensor_info(m->a, i);
    maxn = std::max(maxn, (size_t)(t.rows * t.cols));
  }
  float* staging = nullptr;
  if (dev_malloc((void**)&staging, maxn * sizeof(float)) != cudaSuccess) {
    cudaGetLastError();
    track_model_destroy(m);
    return fail(TRACK_ENOMEM, "staging allocation failed");
  }
  int rc = TRACK_OK;
  for (int i = 0; i < nt && rc == TRACK_OK; ++i) {
    const TensorInfo t = tensor_info(m->a, i);
    const size_t n = (size_t)(t.rows * t.cols);
    cudaError_t e = cudaMemcpy(staging, weights[i], n * sizeof(float), cudaMemcpyHostToDevice);
    if (e == cudaSuccess)
      e = convert_f32(staging, m->tensor_ptr[i], t.matrix ? m->dtype : F32, (int64_t)n, 0);
    if (e == cudaSuccess) e = cudaDeviceSynchronize();
    if (e != cudaSuccess) rc = fail(TRACK_ECUDA, std::string("weight upload: ") + cudaGetErrorString(e));
  }
  cudaFree(staging);
  if (rc != TRACK_OK) {
    track_model_destroy(m);
    return rc;
  }
  *out = m;
  return TRACK_OK;
}


int track_model_create_seeded(const track_arch* arch, uint32_t seed, track_model** out) {
  track_model* m = nullptr;
  TRACK_TRY(model_alloc(arch, out, &m));
  const int nt = n_tensors(m->a);
  for (int i = 0; i < nt; ++i) {
    const TensorInfo t = tensor_info(m->a, i);
    double sigma = 0.02;
    float offset = 0.f;
    int has_offset = 0;
    if (t.kind == 'W') sigma = 1.0 / sqrt((double)t.cols);
    else if (t.kind == 'g') { sigma = 0.05; offset = 1.f; has_offset = 1; }
    else if (t.kind == 'z') sigma = 0.05;
    const float scale = (float)(sigma * sqrt(3.0) / 131072.0);
    const uint64_t state = mix64_host(((uint64_t)seed << 32) | (uint64_t)(uint32_t)i);
    cudaError_t e = seed_fill(m->tensor_ptr[i], t.matrix ? m->dtype : F32, state,
                              (int64_t)(t.rows * t.cols), scale, offset, has_offset, 0);
    if (e != cudaSuccess) {
      track_model_destroy(m);
      return fail(TRACK_ECUDA, std::string("seeded init: ") + cudaGetErrorString(e));
    }
  }
  cudaError_t e = cudaDeviceSynchronize();
  if (e != cudaSuccess) {
    track_model_destroy(m);
    return fail(TRACK_ECUDA, std::string("seeded init: ") + cudaGetErrorString(e));
  }
  *out = m;
  return TRACK_OK;
}

int track_models_compatible(const track_model* a, const track_model* b) {
  if (!a || !b) {
    fail(TRACK_EINVAL, "model is NULL");
    return -1;
  }
  const track_arch &x = a->a, &y = b->a;
  return x.in_ch == y.in_ch && x.frames == y.frames && x.height == y.height && x.width == y.width &&
         x.patch_f == y.patch_f && x.patch_h == y.patch_h && x.patch_w == y.patch_w &&
         x.text_len == y.text_len && x.text_dim == y.text_dim && a->dev == b->dev;
}

int track_invalidate_ctx(track_model* m) {
  if (!m) return fail(TRACK_EINVAL, "model is NULL");
  m->c_valid = false;
  return TRACK_OK;
}

int track_denoise(track_model* m, const float* x_t, int B, float t, const float* cond,
                  const float* uncond, float cfg_scale, float* v_out, track_stream s) {
  TRACK_TRY(check_denoise_args(m, x_t, B, cond, uncond, cfg_scale, v_out));
  if ((const void*)x_t == (const void*)v_out) return fail(TRACK_EINVAL, "v_out aliases x_t");
  TRACK_TRY(set_device(m));
  return denoise_impl(m, x_t, B, t, cond, uncond, cfg_scale, v_out, (cudaStream_t)s);
}

int track_denoise_step(track_model* m, float* x, int B, float sigma_t, float sigma_next,
                       const float* cond, const float* uncond, float cfg_scale, track_stream s) {
  TRACK_TRY(check_denoise_args(m, x, B, cond, uncond, cfg_scale, x));
  TRACK_TRY(set_device(m));
  return denoise_step_impl(m, x, B, sigma_t, sigma_next, cond, uncond, cfg_scale, (cudaStream_t)s);
}

int track_cfg(const float* f_c, const float* f_u, int64_t n, float w, float* p_out, track_stream s) {
  if (n < 0 || !f_c || !p_out || (w != 1.f && !f_u)) return fail(TRACK_EINVAL, "bad arguments");
  LAUNCH(cfg_combine(f_c, f_u, n, w, p_out, (cudaStream_t)s));
  return TRACK_OK;
}

int track_schedule(int n_steps, float shift, float* sigmas_out) {
  if (n_steps < 1 || !(shift > 0.f) || !isfinite(shift) || !sigmas_out)
    return fail(TRACK_EINVAL, "n_steps >= 1, shift > 0 and an output array are required");
  for (int i = 0; i <= n_steps; ++i) {
    const double u = 1.0 - (double)i / (double)n_steps;
    sigmas_out[i] = (float)((double)shift * u / (1.0 + ((double)shift - 1.0) * u));
  }
  return TRACK_OK;
}

int track_step(float* x_t, const float* v, int64_t n, float sigma_t, float sigma_next,
               track_stream s) {
  if (n < 0 || !x_t || !v) return fail(TRACK_EINVAL, "bad arguments");
  LAUNCH(euler_step(x_t, v, n, sigma_next - sigma_t, (cudaStream_t)s));
  return TRACK_OK;
}

int track_cfg_step(float* x, const float* f_c, const float* f_u, int64_t n, float w, float sigma_t,
                   float sigma_next, track_stream s) {
  if (n < 0 || !x || !f_c || (w != 1.f && !f_u)) return fail(TRACK_EINVAL, "bad arguments");
  LAUNCH(cfg_euler(x, f_c, f_u, n, w, sigma_next - sigma_t, (cudaStream_t)s));
  return TRACK_OK;
}

int track_disagreement(const float* v_L, const float* v_S, int B, int64_t n_per_sample, float eps,
                       float* score_accum, track_stream s) {
  if (!v_L || !v_S || !score_accum || B < 0 || n_per_sample <= 0 || !(eps > 0.f))
    return fail(TRACK_EINVAL, "bad arguments");
  if (B == 0) return TRACK_OK;
  return disagreement_impl(v_L, v_S, B, n_per_sample, eps, score_accum, (cudaStream_t)s);
}

int track_disagreement_update(const float* v_L, const float* v_S, int B, int64_t n_per_sample,
                              float eps, float* score_accum, float* x, float sigma_t,
                              float sigma_next, track_stream s) {
  if (!v_L || !v_S || !score_accum || !x || B < 0 || n_per_sample <= 0 || !(eps > 0.f))
    return fail(TRACK_EINVAL, "bad arguments");
  if (B == 0) return TRACK_OK;
  const uintptr_t xb = (uintptr_t)x, xe = xb + (uintptr_t)B * n_per_sample * sizeof(float);
  for (const float* v : {v_L, v_S}) {
    const uintptr_t vb = (uintptr_t)v, ve = vb + (uintptr_t)B * n_per_sample * sizeof(float);
    if (xb < ve && vb < xe) return fail(TRACK_EINVAL, "x overlaps v_L or v_S");
  }
  return disagreement_impl(v_L, v_S, B, n_per_sample, eps, score_accum, (cudaStream_t)s, x,
                           sigma_next - sigma_t);
}

int track_mean_score(const float* r, int M, int N, float* q_out) {
  if (!r || !q_out || M < 1 || N < 1) return fail(TRACK_EINVAL, "bad arguments");
  for (int k = 0; k < N; ++k) {
    double acc = 0.0;
    for (int j = 0; j < M; ++j) acc += (double)r[(size_t)j * N + k];
    q_out[k] = (float)(acc / M);
  }
  return TRACK_OK;
}

static const char kScoreMagic[8] = {'T', 'R', 'K', 'S', 'C', 'O', 'R', 'E'};

// Little-endian encoding independent of the host's byte order.
static void put_u32(std::vector<uint8_t>& b, uint32_t v) {
  for (int i = 0; i < 4; ++i) b.push_back((uint8_t)(v >> (8 * i)));
}
static void put_u64(std::vector<uint8_t>& b, uint64_t v) {
  for (int i = 0; i < 8; ++i) b.push_back((uint8_t)(v >> (8 * i)));
}
static void put_f32(std::vector<uint8_t>& b, float f) {
  uint32_t u;
  memcpy(&u, &f, 4);
  put_u32(b, u);
}
static uint32_t get_u32(const uint8_t* p) {
  uint32_t v = 0;
  for (int i = 0; i < 4; ++i) v |= (uint32_t)p[i] << (8 * i);
  return v;
}
static uint64_t get_u64(const uint8_t* p) {
  uint64_t v = 0;
  for (int i = 0; i < 8; ++i) v |= (uint64_t)p[i] << (8 * i);
  return v;
}
static float get_f32(const uint8_t* p) {
  const uint32_t u = get_u32(p);
  float f;
  memcpy(&f, &u, 4);
  return f;
}

int track_score_map_save(const char* path, const float* r, int M, int N, uint64_t config_hash) {
  if (!path || !r || M < 1 || N < 1) return fail(TRACK_EINVAL, "bad arguments");
  const size_t n = (size_t)M * N;
  for (size_t i = 0; i < n; ++i)
    if (!(r[i] >= 0.f)) return fail(TRACK_EINVAL, "scores must be non-negative numbers");
  std::vector<float> q((size_t)N);
  TRACK_TRY(track_mean_score(r, M, N, q.data()));
  std::vector<uint8_t> b;
  b.reserve(28 + 4 * (n + N));
  b.insert(b.end(), kScoreMagic, kScoreMagic + 8);
  put_u32(b, 1);
  put_u32(b, (uint32_t)M);
  put_u32(b, (uint32_t)N);
  put_u64(b, config_hash);
  for (size_t i = 0; i < n; ++i) put_f32(b, r[i]);
  for (int k = 0; k < N; ++k) put_f32(b, q[(size_t)k]);
  FILE* f = fopen(path, "wb");
  if (!f) return fail(TRACK_EINVAL, std::string("cannot open for writing: ") + path);
  const size_t w = fwrite(b.data(), 1, b.size(), f);
  const int closed = fclose(f);
  if (w != b.size() || closed != 0) return fail(TRACK_EINVAL, std::string("write failed: ") + path);
  return TRACK_OK;
}

int track_score_map_load(const char* path, float* r, int64_t r_cap, float* q, int64_t q_cap,
                         int* M, int* N, uint64_t* config_hash) {
  if (!path || !r || !M || !N || !config_hash || r_cap < 1 || (q && q_cap < 1))
    return fail(TRACK_EINVAL, "bad arguments");
  FILE* f = fopen(path, "rb");
  if (!f) return fail(TRACK_EINVAL, std::string("cannot open: ") + path);
  std::vector<uint8_t> b;
  uint8_t buf[65536];
  size_t got;
  while ((got = fread(buf, 1, sizeof(buf), f)) > 0) b.insert(b.end(), buf, buf + got);
  fclose(f);
  if (b.size() < 28 || memcmp(b.data(), kScoreMagic, 8) != 0)
    return fail(TRACK_EINVAL, "not a score-map file");
  if (get_u32(b.data() + 8) != 1) return fail(TRACK_EINVAL, "unknown score-map version");
  const uint32_t m = get_u32(b.data() + 12), n = get_u32(b.data() + 16);
  if (m < 1 || n < 1 || m > (1u << 30) || n > (1u << 30)) return fail(TRACK_EINVAL, "bad dimensions");
  const uint64_t need = 28 + 4 * ((uint64_t)m * n + n);
  if ((uint64_t)b.size() != need) return fail(TRACK_EINVAL, "truncated or oversized score-map file");
  if ((int64_t)m * n > r_cap || (q && (int64_t)n > q_cap))
    return fail(TRACK_EINVAL, "score map larger than the given capacity");
  const uint8_t* p = b.data() + 28;
  for (uint64_t i = 0; i < (uint64_t)m * n; ++i) r[i] = get_f32(p + 4 * i);
  if (q)
    for (uint32_t k = 0; k < n; ++k) q[k] = get_f32(p + 4 * ((uint64_t)m * n + k));
  *M = (int)m;
  *N = (int)n;
  *config_hash = get_u64(b.data() + 20);
  return TRACK_OK;
}

int track_policy_topk(const float* score_map, int N, int K, uint8_t* policy_out) {
  if (!score_map || !policy_out || N < 1) return fail(TRACK_EINVAL, "bad arguments");
  if (K < 0 || K > N) return fail(TRACK_EINVAL, "K must satisfy 0 <= K <= N");
  for (int i = 0; i < N; ++i)
    if (!(score_map[i] >= 0.f)) return fail(TRACK_EINVAL, "scores must be non-negative numbers");
  std::vector<int> idx(N);
  for (int i = 0; i < N; ++i) idx[i] = i;
  std::stable_sort(idx.begin(), idx.end(),
                   [&](int a, int b) { return score_map[a] < score_map[b]; });
  for (int i = 0; i < N; ++i) policy_out[i] = 0;
  for (int i = 0; i < K; ++i) policy_out[idx[i]] = 1;
  return TRACK_OK;
}

int track_policy_first_k(int N, int K, uint8_t* policy_out) {
  if (!policy_out || N < 1 || K < 0 || K > N) return fail(TRACK_EINVAL, "bad arguments");
  for (int i = 0; i < N; ++i) policy_out[i] = i < K ? 1 : 0;
  return TRACK_OK;
}

int track_policy_last_k(int N, int K, uint8_t* policy_out) {
  if (!policy_out || N < 1 || K < 0 || K > N) return fail(TRACK_EINVAL, "bad arguments");
  for (int i = 0; i < N; ++i) policy_out[i] = i >= N - K ? 1 : 0;
  return TRACK_OK;
}

int track_policy_random_k(int N, int K, uint64_t seed, uint8_t* policy_out) {
  if (!policy_out || N < 1 || K < 0 || K > N) return fail(TRACK_EINVAL, "bad arguments");
  std::vector<int> perm(N);
  for (int i = 0; i < N; ++i) perm[i] = i;
  const uint64_t state = mix64_host(seed);
  for (int i = 0; i < K; ++i) {
    const uint64_t u = mix64_host(state + (uint64_t)(i + 1) * 0x9E3779B97F4A7C15ull);
    const int j = i + (int)(u % (uint64_t)(N - i));
    std::swap(perm[i], perm[j]);
  }
  for (int i = 0; i < N; ++i) policy_out[i] = 0;
  for (int i = 0; i < K; ++i) policy_out[perm[i]] = 1;
  return TRACK_OK;
}

int track_calibrate(track_model* large, track_model* small, float* x, int B, const float* cond,
                    const float* uncond, float cfg_scale, const float* sigmas, int n_steps,
                    float eps, float* r_out, track_stream s) {
  if (!large || !small) return fail(TRACK_EINVAL, "model is NULL");
  if (track_models_compatible(large, small) != 1)
    return fail(TRACK_EINVAL, "models are not a compatible pair");
  if (!sigmas || !r_out || n_steps < 1 || !(eps > 0.f)) return fail(TRACK_EINVAL, "bad arguments");
  TRACK_TRY(check_denoise_args(large, x, B, cond, uncond, cfg_scale, x));
  TRACK_TRY(set_device(large));
  cudaStream_t st = (cudaStream_t)s;
  TRACK_TRY(ensure_calib(large, B));
  float* pL = large->ws.pL;
  float* pS = large->ws.pS;
  const int64_t n = large->latent_n;
  TRACK_CUDA(cudaMemsetAsync(r_out, 0, (size_t)n_steps * B * sizeof(float), st));
  for (int k = 0; k < n_steps; ++k) {
    const float t = 1000.f * sigmas[k];
    TRACK_TRY(denoise_impl(large, x, B, t, cond, uncond, cfg_scale, pL, st));
    TRACK_TRY(denoise_impl(small, x, B, t, cond, uncond, cfg_scale, pS, st));
    // Eq. 4 and the trajectory's Euler update by p_L in one pass
    TRACK_TRY(disagreement_impl(pL, pS, B, n, eps, r_out + (size_t)k * B, st, x,
                                sigmas[k + 1] - sigmas[k]));
  }
  return TRACK_OK;
}

int track_sample(track_model* large, track_model* small, const uint8_t* policy, const float* sigmas,
                 int n_steps, float* x, int B, const float* cond, const float* uncond,
                 float cfg_scale, track_stream s) {
  if (!large || !small) return fail(TRACK_EINVAL, "model is NULL");
  if (track_models_compatible(large, small) != 1)
    return fail(TRACK_EINVAL, "models are not a compatible pair");
  if (!policy || !sigmas || n_steps < 1) return fail(TRACK_EINVAL, "bad arguments");
  TRACK_TRY(check_denoise_args(large, x, B, cond, uncond, cfg_scale, x));
  TRACK_TRY(set_device(large));
  for (int i = 0; i < n_steps; ++i) {
    track_model* m = policy[i] ? small : large;
    TRACK_TRY(denoise_step_impl(m, x, B, sigmas[i], sigmas[i + 1], cond, uncond, cfg_scale,
                                (cudaStream_t)s));
  }
  return TRACK_OK;
}

// ---------------------------------------------------------------- routed loop as a CUDA graph
namespace {
struct GraphEntry {
  track_model *L, *S;
  std::string policy;
  std::vector<float> sigmas;
  float* x;
  int B;
  const float *cond, *uncond;
  float w;
  cudaStream_t s;
  int dev;
  uint64_t gen_L, gen_S, gen_sk;  // allocations the graph's addresses come from
  bool prof = false;                 // recorded with profiling on: bracketed launches
  cudaGraphExec_t exec = nullptr;
  int64_t launches = 0;              // kernels recorded in the graph
  std::vector<ProfRec> recs;         // the brackets' events (prof graphs only)
};
std::mutex g_graph_mu;
std::vector<GraphEntry> g_graphs;
constexpr size_t kMaxGraphs = 32;

bool same_call(const GraphEntry& e, const GraphEntry& k) {
  return e.L == k.L && e.S == k.S && e.policy == k.policy && e.sigmas == k.sigmas && e.x == k.x &&
         e.B == k.B && e.cond == k.cond && e.uncond == k.uncond && e.w == k.w && e.s == k.s &&
         e.dev == k.dev && e.prof == k.prof;
}

// Destroys the executable graph and the events of its brackets; brackets of
// its replays that were not read yet are discarded.
void drop_graph(GraphEntry& e) {
  if (e.exec) cudaGraphExecDestroy(e.exec);
  e.exec = nullptr;
  if (e.recs.empty()) return;
  {
    std::lock_guard<std::mutex> lk(g_prof_mu);
    std::unordered_set<cudaEvent_t> mine;
    for (const ProfRec& r : e.recs) mine.insert(r.a);
    g_prof.erase(std::remove_if(g_prof.begin(), g_prof.end(),
                                [&mine](const ProfRec& q) { return mine.count(q.a) != 0; }),
                 g_prof.end());
  }
  for (const ProfRec& r : e.recs) {
    cudaEventDestroy(r.a);
    cudaEventDestroy(r.b);
  }
  e.recs.clear();
}

// The routed loop of Eq. 3 with the text projection always recomputed.
int sample_loop(track_model* large, track_model* small, const uint8_t* policy,
                const float* sigmas, int n_steps, float* x, int B, const float* cond,
                const float* uncond, float cfg_scale, cudaStream_t s) {
  large->c_valid = false;
  small->c_valid = false;
  for (int i = 0; i < n_steps; ++i) {
    track_model* m = policy[i] ? small : large;
    TRACK_TRY(denoise_step_impl(m, x, B, sigmas[i], sigmas[i + 1], cond, uncond, cfg_scale, s));
  }
  return TRACK_OK;
}
}  // namespace

// Drops every recorded graph that uses model m.
static void drop_graphs_of(const track_model* m) {
  std::lock_guard<std::mutex> lk(g_graph_mu);
  for (size_t i = 0; i < g_graphs.size();) {
    if (g_graphs[i].L == m || g_graphs[i].S == m) {
      drop_graph(g_graphs[i]);
      g_graphs.erase(g_graphs.begin() + (long)i);
    } else {
      ++i;
    }
  }
}

int track_band_disagreement(const float* v_L, const float* v_S, int B, int C, int F, int H, int W,
                            float eps, float* bands_out, track_stream s) {
  if (!v_L || !v_S || !bands_out) return fail(TRACK_EINVAL, "NULL pointer");
  if (B < 0 || C <= 0 || F <= 0 || H <= 0 || W <= 0) return fail(TRACK_EINVAL, "bad shape");
  if (F > 512 || H > 512 || W > 512) return fail(TRACK_EUNSUPPORTED, "axes longer than 512");
  if (!(eps >= 0.f)) return fail(TRACK_EINVAL, "eps must be non-negative");
  return band_impl(v_L, v_S, B, C, F, H, W, eps, bands_out, (cudaStream_t)s);
}

int track_multistep_step(float* x, const float* v, float* state, int64_t n, const float* sigmas,
                         int n_steps, int i, track_stream s) {
  if (!x || !v || !state || !sigmas) return fail(TRACK_EINVAL, "NULL pointer");
  if (n < 0 || n_steps < 1 || i < 0 || i >= n_steps) return fail(TRACK_EINVAL, "bad step index");
  if ((((uintptr_t)x) | ((uintptr_t)v) | ((uintptr_t)state)) & 15)
    return fail(TRACK_EINVAL, "device pointers must be 16-byte aligned");
  if (v == x || v == state || v == state + n) return fail(TRACK_EINVAL, "v may not alias x or state");
  LAUNCH(multistep_step(x, v, state, state + n, n, sigmas, i, (cudaStream_t)s));
  return TRACK_OK;
}

int track_sample_multistep(track_model* large, track_model* small, const uint8_t* policy,
                           const float* sigmas, int n_steps, float* x, int B, const float* cond,
                           const float* uncond, float cfg_scale, float* state, track_stream s) {
  if (!large || !small) return fail(TRACK_EINVAL, "model is NULL");
  if (track_models_compatible(large, small) != 1)
    return fail(TRACK_EINVAL, "models are not a compatible pair");
  if (!policy || !sigmas || n_steps < 1 || !state) return fail(TRACK_EINVAL, "bad arguments");
  if (((uintptr_t)state) & 15) return fail(TRACK_EINVAL, "state must be 16-byte aligned");
  TRACK_TRY(check_denoise_args(large, x, B, cond, uncond, cfg_scale, x));
  TRACK_TRY(set_device(large));
  const cudaStream_t st = (cudaStream_t)s;
  const int64_t n = (int64_t)B * large->latent_n;
  const int nseq = cfg_scale == 1.f ? B : 2 * B;
  for (int i = 0; i < n_steps; ++i) {
    track_model* m = policy[i] ? small : large;
    TRACK_TRY(ensure_workspace(m, nseq));
    float* p = m->ws.fout;
    TRACK_TRY(forward(m, x, B, nseq, 1000.f * sigmas[i], cond, cfg_scale == 1.f ? nullptr : uncond,
                      p, st));
    if (cfg_scale != 1.f) LAUNCH(cfg_combine(p, p + n, n, cfg_scale, p, st));  // in place
    LAUNCH(multistep_step(x, p, state, state + n, n, sigmas, i, st));
  }
  return TRACK_OK;
}

int track_sample_graph(track_model* large, track_model* small, const uint8_t* policy,
                       const float* sigmas, int n_steps, float* x, int B, const float* cond,
                       const float* uncond, float cfg_scale, track_stream s) {
  if (!large || !small) return fail(TRACK_EINVAL, "model is NULL");
  if (track_models_compatible(large, small) != 1)
    return fail(TRACK_EINVAL, "models are not a compatible pair");
  if (!policy || !sigmas || n_steps < 1) return fail(TRACK_EINVAL, "bad arguments");
  if ((cudaStream_t)s == nullptr || (cudaStream_t)s == cudaStreamLegacy)
    return fail(TRACK_EINVAL, "a CUDA graph cannot be recorded on the legacy default stream");
  TRACK_TRY(check_denoise_args(large, x, B, cond, uncond, cfg_scale, x));
  TRACK_TRY(set_device(large));
  const cudaStream_t st = (cudaStream_t)s;
  GraphEntry key;
  key.L = large; key.S = small;
  key.policy.assign((const char*)policy, (size_t)n_steps);
  key.sigmas.assign(sigmas, sigmas + n_steps + 1);
  key.x = x; key.B = B; key.cond = cond; key.uncond = cfg_scale == 1.f ? nullptr : uncond;
  key.w = cfg_scale; key.s = st; key.dev = large->dev;
  key.prof = g_prof_on.load(std::memory_order_relaxed);
  cudaGraphExec_t exec = nullptr;
  int64_t nlaunch = 0;
  bool warm = false;
  std::vector<ProfRec> recs;
  {
    std::lock_guard<std::mutex> lk(g_graph_mu);
    for (size_t i = 0; i < g_graphs.size(); ++i) {
      GraphEntry& e = g_graphs[i];
      if (!same_call(e, key)) continue;
      if (e.gen_L != large->ws_gen || e.gen_S != small->ws_gen ||
          e.gen_sk != sk_scratch_generation()) {  // an address it holds was freed
        drop_graph(e);
        g_graphs.erase(g_graphs.begin() + (long)i);
        break;
      }
      warm = true;
      exec = e.exec;
      nlaunch = e.launches;
      recs = e.recs;
      break;
    }
  }
  if (!warm) {
    // First call with these arguments: run eagerly, which also sizes every
    // buffer the graph will address.
    TRACK_TRY(sample_loop(large, small, policy, sigmas, n_steps, x, B, cond, uncond, cfg_scale, st));
    key.gen_L = large->ws_gen;
    key.gen_S = small->ws_gen;
    key.gen_sk = sk_scratch_generation();
    std::lock_guard<std::mutex> lk(g_graph_mu);
    if (g_graphs.size() >= kMaxGraphs) {
      drop_graph(g_graphs.front());
      g_graphs.erase(g_graphs.begin());
    }
    g_graphs.push_back(key);
    return TRACK_OK;
  }
  if (exec == nullptr) {
    // Second call: record the loop (kernels are recorded, not run) and instantiate it.
    cudaGraph_t graph = nullptr;
    TRACK_CUDA(cudaStreamBeginCapture(st, cudaStreamCaptureModeThreadLocal));
    g_capturing = true;
    g_capture_recs = key.prof ? &recs : nullptr;
    const int64_t n0 = track_launch_count();
    const int rc =
        sample_loop(large, small, policy, sigmas, n_steps, x, B, cond, uncond, cfg_scale, st);
    nlaunch = track_launch_count() - n0;
    g_capturing = false;
    g_capture_recs = nullptr;
    const cudaError_t ce = cudaStreamEndCapture(st, &graph);
    large->c_valid = small->c_valid = false;  // the recorded projection has not run yet
    auto free_recs = [&recs]() {
      for (const ProfRec& r : recs) {
        cudaEventDestroy(r.a);
        cudaEventDestroy(r.b);
      }
      recs.clear();
    };
    if (rc != TRACK_OK) {
      if (graph) cudaGraphDestroy(graph);
      free_recs();
      return rc;
    }
    if (ce != cudaSuccess) {
      free_recs();
      return fail(TRACK_ECUDA, std::string("graph capture: ") + cudaGetErrorString(ce));
    }
    const cudaError_t ie = cudaGraphInstantiate(&exec, graph, 0);
    cudaGraphDestroy(graph);
    if (ie != cudaSuccess) {
      free_recs();
      return fail(TRACK_ECUDA, std::string("graph instantiate: ") + cudaGetErrorString(ie));
    }
    g_launches.fetch_sub(nlaunch, std::memory_order_relaxed);  // recorded, not launched
    std::lock_guard<std::mutex> lk(g_graph_mu);
    bool stored = false;
    for (GraphEntry& e : g_graphs)
      if (!stored && same_call(e, key)) {
        e.exec = exec;
        e.launches = nlaunch;
        e.recs = recs;
        stored = true;
      }
    if (!stored) {  // evicted meanwhile: keep the recording under a fresh entry
      key.gen_L = large->ws_gen;
      key.gen_S = small->ws_gen;
      key.gen_sk = sk_scratch_generation();
      key.exec = exec;
      key.launches = nlaunch;
      key.recs = recs;
      if (g_graphs.size() >= kMaxGraphs) {
        drop_graph(g_graphs.front());
        g_graphs.erase(g_graphs.begin());
      }
      g_graphs.push_back(key);
    }
  }
  TRACK_CUDA(cudaGraphLaunch(exec, st));
  count_launch((int)nlaunch);
  if (!recs.empty()) {
    // Every replay re-records the same events: the brackets hold the latest
    // replay until read.
    std::lock_guard<std::mutex> lk(g_prof_mu);
    std::unordered_set<cudaEvent_t> pending;
    for (const ProfRec& q : g_prof) pending.insert(q.a);
    for (const ProfRec& r : recs)
      if (pending.count(r.a) == 0) g_prof.push_back(r);
  }
  return TRACK_OK;
}

int track_linear(int dtype, const void* X, const void* W, const float* bias, int M, int N, int K,
                 int epilogue, const float* gate, void* out, int ldo, track_stream s) {
  if (!X || !W || !out || M < 0 || N <= 0 || K <= 0 || ldo < N)
    return fail(TRACK_EINVAL, "bad arguments");
  if (epilogue < 0 || epilogue > 3) return fail(TRACK_EINVAL, "bad epilogue");
  if (epilogue == TRACK_EPI_RESID_GATE && !gate) return fail(TRACK_EINVAL, "gate is NULL");
  if (dtype == TRACK_BF16 && (K % 64 || N % 32 || ldo % 8))
    return fail(TRACK_EUNSUPPORTED, "bf16 GEMM needs K % 64 == 0, N % 32 == 0, ldo % 8 == 0");
  GemmArgs g;
  g.M = M; g.N = N; g.K = K; g.epi = epilogue; g.bias = bias; g.gate = gate; g.out = out;
  g.ldo = ldo; g.err = device_error_word();
  if (!g.err) return fail(TRACK_ECUDA, "device error word");
  cudaError_t e = dtype == TRACK_BF16 ? gemm_bf16_tc(X, W, g, (cudaStream_t)s)
                                      : gemm_f32((const float*)X, (const float*)W, g, (cudaStream_t)s);
  if (e != cudaSuccess) return fail(TRACK_ECUDA, std::string("gemm: ") + cudaGetErrorString(e));
  return TRACK_OK;
}

int track_attention(int dtype, const void* Q, const void* K, const void* V, int S, int H, int Lq,
                    int Lk, int hd, void* O, track_stream s) {
  if (!Q || !K || !V || !O || S < 0 || H <= 0 || Lq < 0 || Lk <= 0)
    return fail(TRACK_EINVAL, "bad arguments");
  if (hd != 64 && hd != 128) return fail(TRACK_EINVAL, "hd must be 64 or 128");
  const AttnOperand q = head_major(Q, H, Lq, hd), k = head_major(K, H, Lk, hd),
                    v = head_major(V, H, Lk, hd);
  cudaError_t e = dtype == TRACK_BF16
                      ? attention_bf16(q, k, v, O, S, H, Lq, Lk, hd, (cudaStream_t)s)
                      : attention_f32(q, k, v, (float*)O, S, H, Lq, Lk, hd, (cudaStream_t)s);
  if (e != cudaSuccess) return fail(TRACK_ECUDA, std::string("attention: ") + cudaGetErrorString(e));
  return TRACK_OK;
}

}  // extern "C"
