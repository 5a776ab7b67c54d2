"""GB300 (sm_103a) implementation of TRACK's routed denoising hot path.

This package is a thin ctypes binding over ``libtrack.so`` (built from
``csrc/`` by ``_build.build()``), whose C ABI is declared in
``include/track.h``.  Every function below marshals arguments and calls the
C entry point of the same name; every step of the computation runs in the
library's CUDA kernels.  Torch tensors are used only as device memory and
the current CUDA stream.  There is no fallback: if the library is missing or
fails to load, calls raise.
"""
from __future__ import annotations

import ctypes
import os

import numpy as np

from ._build import LIB as _LIB_PATH

TRACK_OK, TRACK_EINVAL, TRACK_ENOMEM, TRACK_ECUDA, TRACK_EUNSUPPORTED, TRACK_ETIMEOUT = range(6)
TRACK_WAIT_SELFTEST_CODE = 99  # error-word code of track_wait_selftest
FP32, BF16 = 0, 1
EPI_STORE, EPI_GELU, EPI_RESID_GATE, EPI_RESID = range(4)
GEMM_AUTO, GEMM_DATA_PARALLEL, GEMM_STREAM_K = range(3)
ATTN_ONE_TILE = 4   # OR-ed into an attention schedule: one query tile per work item


class TrackError(RuntimeError):
    def __init__(self, code, msg):
        super().__init__(f"[{code}] {msg}")
        self.code = code


class ArchC(ctypes.Structure):
    _fields_ = [(n, ctypes.c_int) for n in (
        "dim", "layers", "heads", "ffn", "text_dim", "text_len", "in_ch", "frames", "height",
        "width", "patch_f", "patch_h", "patch_w", "freq_dim", "dtype")] + [("eps", ctypes.c_float)]


_lib = None
_P = ctypes.c_void_p
_I = ctypes.c_int
_L = ctypes.c_int64
_F = ctypes.c_float


def lib():
    """The loaded libtrack (raises if it has not been built)."""
    global _lib
    if _lib is not None:
        return _lib
    if not os.path.exists(_LIB_PATH):
        raise RuntimeError(f"{_LIB_PATH} is missing: build it with __graft_entry__.build() "
                           "(the CUDA library is required; there is no fallback)")
    L = ctypes.CDLL(_LIB_PATH)
    sig = {
        "track_last_error": (ctypes.c_char_p, []),
        "track_abi_version": (_I, []),
        "track_sync": (_I, [_P]),
        "track_launch_count": (_L, []),
        "track_profile_enable": (_I, [_I]),
        "track_gemm_schedule": (_I, [_I]),
        "track_attention_schedule": (_I, [_I]),
        "track_gemm_raster": (_I, [_I]),
        "track_score_map_save": (_I, [ctypes.c_char_p, _P, _I, _I, ctypes.c_uint64]),
        "track_score_map_load": (_I, [ctypes.c_char_p, _P, ctypes.c_int64, _P, ctypes.c_int64,
                                      ctypes.POINTER(_I), ctypes.POINTER(_I),
                                      ctypes.POINTER(ctypes.c_uint64)]),
        "track_wait_selftest": (_I, [ctypes.c_int64, _P]),
        "track_fail_next_allocations": (_I, [_I]),
        "track_profile_read": (_I, [_P, _P, _P]),
        "track_weight_count": (_I, [_P]),
        "track_weight_shape": (_I, [_P, _I, _P, _P]),
        "track_model_create": (_I, [_P, _P, _P]),
        "track_model_create_seeded": (_I, [_P, ctypes.c_uint32, _P]),
        "track_model_destroy": (_I, [_P]),
        "track_models_compatible": (_I, [_P, _P]),
        "track_invalidate_ctx": (_I, [_P]),
        "track_denoise": (_I, [_P, _P, _I, _F, _P, _P, _F, _P, _P]),
        "track_denoise_step": (_I, [_P, _P, _I, _F, _F, _P, _P, _F, _P]),
        "track_cfg": (_I, [_P, _P, _L, _F, _P, _P]),
        "track_schedule": (_I, [_I, _F, _P]),
        "track_step": (_I, [_P, _P, _L, _F, _F, _P]),
        "track_cfg_step": (_I, [_P, _P, _P, _L, _F, _F, _F, _P]),
        "track_disagreement": (_I, [_P, _P, _I, _L, _F, _P, _P]),
        "track_disagreement_update": (_I, [_P, _P, _I, _L, _F, _P, _P, _F, _F, _P]),
        "track_disagreement_static": (_I, [_P, _P, _I, _L, _F, _P, _P]),
        "track_mean_score": (_I, [_P, _I, _I, _P]),
        "track_policy_topk": (_I, [_P, _I, _I, _P]),
        "track_policy_first_k": (_I, [_I, _I, _P]),
        "track_policy_last_k": (_I, [_I, _I, _P]),
        "track_policy_random_k": (_I, [_I, _I, ctypes.c_uint64, _P]),
        "track_calibrate": (_I, [_P, _P, _P, _I, _P, _P, _F, _P, _I, _F, _P, _P]),
        "track_sample": (_I, [_P, _P, _P, _P, _I, _P, _I, _P, _P, _F, _P]),
        "track_sample_graph": (_I, [_P, _P, _P, _P, _I, _P, _I, _P, _P, _F, _P]),
        "track_multistep_step": (_I, [_P, _P, _P, ctypes.c_int64, _P, _I, _I, _P]),
        "track_band_disagreement": (_I, [_P, _P, _I, _I, _I, _I, _I, _F, _P, _P]),
        "track_sample_multistep": (_I, [_P, _P, _P, _P, _I, _P, _I, _P, _P, _F, _P, _P]),
        "track_linear": (_I, [_I, _P, _P, _P, _I, _I, _I, _I, _P, _P, _I, _P]),
        "track_attention": (_I, [_I, _P, _P, _P, _I, _I, _I, _I, _I, _P, _P]),
    }
    for name, (res, args) in sig.items():
        f = getattr(L, name)
        f.restype = res
        f.argtypes = args
    _lib = L
    return L


def _check(rc):
    if rc != TRACK_OK:
        raise TrackError(rc, lib().track_last_error().decode())


def arch_c(arch, dtype=FP32) -> ArchC:
    """C struct of an architecture object (any object with the ``synth.Arch`` fields)."""
    return ArchC(arch.dim, arch.layers, arch.heads, arch.ffn, arch.text_dim, arch.text_len,
                 arch.in_ch, arch.frames, arch.height, arch.width, *arch.patch, arch.freq_dim,
                 int(dtype), float(arch.eps))


def _ptr(t):
    if t is None:
        return None
    return ctypes.c_void_p(t.data_ptr())


def _stream(stream):
    if stream is not None:
        return ctypes.c_void_p(stream)
    import torch
    return ctypes.c_void_p(torch.cuda.current_stream().cuda_stream)


def _dev_f32(t, name):
    if t is None:
        return
    if not (t.is_cuda and t.is_contiguous()) or str(t.dtype) != "torch.float32":
        raise ValueError(f"{name} must be a contiguous float32 CUDA tensor")


# ---------------------------------------------------------------- library
def track_last_error() -> str:
    return lib().track_last_error().decode()


def track_abi_version() -> int:
    return lib().track_abi_version()


def track_sync(stream=None):
    _check(lib().track_sync(_stream(stream)))


def track_launch_count() -> int:
    return lib().track_launch_count()


def track_gemm_schedule(mode: int):
    """GEMM_AUTO, GEMM_DATA_PARALLEL or GEMM_STREAM_K for every later bf16 GEMM."""
    _check(lib().track_gemm_schedule(int(mode)))


def track_wait_selftest(limit_cycles: int, stream=None):
    """Launches a bounded pipeline wait that is made to run out; the next track_sync
    raises TrackError(TRACK_ETIMEOUT) naming TRACK_WAIT_SELFTEST_CODE."""
    _check(lib().track_wait_selftest(int(limit_cycles), _stream(stream)))


def track_fail_next_allocations(n: int):
    """The next n device allocations of the library fail as out-of-memory (0 clears)."""
    _check(lib().track_fail_next_allocations(int(n)))


def track_gemm_raster(group: int):
    """Row units per raster group of every later bf16 GEMM (0: the default)."""
    _check(lib().track_gemm_raster(int(group)))


def track_attention_schedule(mode: int):
    """GEMM_AUTO, GEMM_DATA_PARALLEL or GEMM_STREAM_K (optionally | ATTN_ONE_TILE) for
    every later bf16 attention."""
    _check(lib().track_attention_schedule(int(mode)))


def track_profile_enable(enable: bool):
    _check(lib().track_profile_enable(int(bool(enable))))


PROFILE_CLASSES = ("gemm", "attention", "layernorm", "norm_rope", "update", "disagreement",
                   "cross_attention")


def track_profile_read():
    """{class: (ms, work, launches)} since the last read, for the classes of
    PROFILE_CLASSES; work is FLOPs for gemm and the attention classes, bytes for the rest."""
    k = len(PROFILE_CLASSES)
    ms = (ctypes.c_double * k)()
    fl = (ctypes.c_double * k)()
    n = (ctypes.c_int64 * k)()
    _check(lib().track_profile_read(ms, fl, n))
    return {c: (ms[i], fl[i], n[i]) for i, c in enumerate(PROFILE_CLASSES)}


# ---------------------------------------------------------------- models
def track_weight_count(arch, dtype=FP32) -> int:
    a = arch_c(arch, dtype)
    n = lib().track_weight_count(ctypes.byref(a))
    if n < 0:
        raise TrackError(TRACK_EINVAL, track_last_error())
    return n


def track_weight_shape(arch, index: int, dtype=FP32):
    a = arch_c(arch, dtype)
    r, c = ctypes.c_int64(), ctypes.c_int64()
    _check(lib().track_weight_shape(ctypes.byref(a), index, ctypes.byref(r), ctypes.byref(c)))
    return r.value, c.value


class Model:
    """Owner of a track_model handle (destroyed with the object)."""

    def __init__(self, handle, arch, dtype):
        self.handle = handle
        self.arch = arch
        self.dtype = dtype

    @property
    def _as_parameter_(self):
        return self.handle

    def close(self):
        if self.handle:
            lib().track_model_destroy(self.handle)
            self.handle = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass


def track_model_create(arch, weights, dtype=FP32) -> Model:
    """weights: sequence of fp32 host arrays in canonical order (e.g. synth.make_weights values)."""
    a = arch_c(arch, dtype)
    arrs = [np.ascontiguousarray(w, dtype=np.float32) for w in weights]
    if len(arrs) != track_weight_count(arch, dtype):
        raise ValueError("wrong number of weight tensors")
    for i, w in enumerate(arrs):
        r, c = track_weight_shape(arch, i, dtype)
        if w.size != r * c:
            raise ValueError(f"weight {i} has {w.size} elements, expected {r}x{c}")
    ptrs = (ctypes.c_void_p * len(arrs))(*[w.ctypes.data for w in arrs])
    h = ctypes.c_void_p()
    _check(lib().track_model_create(ctypes.byref(a), ptrs, ctypes.byref(h)))
    return Model(h, arch, dtype)


def track_model_create_seeded(arch, seed: int, dtype=FP32) -> Model:
    a = arch_c(arch, dtype)
    h = ctypes.c_void_p()
    _check(lib().track_model_create_seeded(ctypes.byref(a), seed, ctypes.byref(h)))
    return Model(h, arch, dtype)


def track_model_destroy(m: Model):
    m.close()


def track_models_compatible(a: Model, b: Model) -> bool:
    r = lib().track_models_compatible(a.handle, b.handle)
    if r < 0:
        raise TrackError(TRACK_EINVAL, track_last_error())
    return r == 1


def track_invalidate_ctx(m: Model):
    _check(lib().track_invalidate_ctx(m.handle))


# ---------------------------------------------------------------- denoiser / guidance / scheduler
def track_denoise(m: Model, x_t, t: float, cond, uncond, cfg_scale: float, v_out=None, stream=None):
    import torch
    for n, v in (("x_t", x_t), ("cond", cond), ("uncond", uncond), ("v_out", v_out)):
        _dev_f32(v, n)
    if v_out is None:
        v_out = torch.empty_like(x_t)
    _check(lib().track_denoise(m.handle, _ptr(x_t), x_t.shape[0], t, _ptr(cond), _ptr(uncond),
                               cfg_scale, _ptr(v_out), _stream(stream)))
    return v_out


def track_denoise_step(m: Model, x, sigma_t, sigma_next, cond, uncond, cfg_scale, stream=None):
    for n, v in (("x", x), ("cond", cond), ("uncond", uncond)):
        _dev_f32(v, n)
    _check(lib().track_denoise_step(m.handle, _ptr(x), x.shape[0], sigma_t, sigma_next, _ptr(cond),
                                    _ptr(uncond), cfg_scale, _stream(stream)))
    return x


def track_cfg(f_c, f_u, w, p_out=None, stream=None):
    import torch
    if p_out is None:
        p_out = torch.empty_like(f_c)
    _check(lib().track_cfg(_ptr(f_c), _ptr(f_u), f_c.numel(), w, _ptr(p_out), _stream(stream)))
    return p_out


def track_schedule(n_steps: int, shift: float) -> np.ndarray:
    out = np.zeros(n_steps + 1, dtype=np.float32)
    _check(lib().track_schedule(n_steps, shift, out.ctypes.data))
    return out


def track_step(x_t, v, sigma_t, sigma_next, stream=None):
    _check(lib().track_step(_ptr(x_t), _ptr(v), x_t.numel(), sigma_t, sigma_next, _stream(stream)))
    return x_t


def track_cfg_step(x, f_c, f_u, w, sigma_t, sigma_next, stream=None):
    _check(lib().track_cfg_step(_ptr(x), _ptr(f_c), _ptr(f_u), x.numel(), w, sigma_t, sigma_next,
                                _stream(stream)))
    return x


# ---------------------------------------------------------------- score and policy
def track_disagreement(v_L, v_S, score_accum, eps=1e-8, stream=None):
    B = v_L.shape[0]
    _check(lib().track_disagreement(_ptr(v_L), _ptr(v_S), B, v_L.numel() // B, eps,
                                    _ptr(score_accum), _stream(stream)))
    return score_accum


def track_disagreement_update(v_L, v_S, score_accum, x, sigma_t, sigma_next, eps=1e-8,
                              stream=None):
    """Eq. 4 into score_accum and the calibration trajectory's Euler update
    x += (sigma_next - sigma_t) * v_L, in one pass (x: same shape as v_L)."""
    B = v_L.shape[0]
    _check(lib().track_disagreement_update(_ptr(v_L), _ptr(v_S), B, v_L.numel() // B, eps,
                                           _ptr(score_accum), _ptr(x), float(sigma_t),
                                           float(sigma_next), _stream(stream)))
    return score_accum


def track_disagreement_static(v_L, v_S, score_accum, eps=1e-8, stream=None):
    """track_disagreement with library-held scratch: allocates no device memory
    (at most 64 samples per call; calls that overlap on the GPU race)."""
    B = v_L.shape[0]
    _check(lib().track_disagreement_static(_ptr(v_L), _ptr(v_S), B, v_L.numel() // B, eps,
                                           _ptr(score_accum), _stream(stream)))
    return score_accum


def track_mean_score(r) -> np.ndarray:
    r = np.ascontiguousarray(r, dtype=np.float32)
    q = np.zeros(r.shape[1], dtype=np.float32)
    _check(lib().track_mean_score(r.ctypes.data, r.shape[0], r.shape[1], q.ctypes.data))
    return q


def track_score_map_save(path, r, config_hash: int = 0):
    """Writes the calibration map r [M, N] (and its Eq. 5 mean) to path."""
    r = np.ascontiguousarray(r, dtype=np.float32)
    if r.ndim != 2:
        raise TrackError(TRACK_EINVAL, "r must be [M, N]")
    _check(lib().track_score_map_save(os.fsencode(path), r.ctypes.data, r.shape[0], r.shape[1],
                                      int(config_hash)))


def track_score_map_load(path):
    """(r [M, N], q [N], config_hash) read from a score-map file."""
    cap = max(1, (os.path.getsize(path) - 28) // 4) if os.path.exists(path) else 1
    r = np.empty(cap, np.float32)
    q = np.empty(cap, np.float32)
    M, N, h = _I(), _I(), ctypes.c_uint64()
    _check(lib().track_score_map_load(os.fsencode(path), r.ctypes.data, cap, q.ctypes.data, cap,
                                      ctypes.byref(M), ctypes.byref(N), ctypes.byref(h)))
    return r[:M.value * N.value].reshape(M.value, N.value).copy(), q[:N.value].copy(), h.value


def track_policy_topk(score_map, K: int) -> np.ndarray:
    q = np.ascontiguousarray(score_map, dtype=np.float32)
    out = np.zeros(q.shape[0], dtype=np.uint8)
    _check(lib().track_policy_topk(q.ctypes.data, q.shape[0], K, out.ctypes.data))
    return out


def track_policy_first_k(N: int, K: int) -> np.ndarray:
    out = np.zeros(N, dtype=np.uint8)
    _check(lib().track_policy_first_k(N, K, out.ctypes.data))
    return out


def track_policy_last_k(N: int, K: int) -> np.ndarray:
    out = np.zeros(N, dtype=np.uint8)
    _check(lib().track_policy_last_k(N, K, out.ctypes.data))
    return out


def track_policy_random_k(N: int, K: int, seed: int) -> np.ndarray:
    out = np.zeros(N, dtype=np.uint8)
    _check(lib().track_policy_random_k(N, K, seed, out.ctypes.data))
    return out


# ---------------------------------------------------------------- loops
def track_calibrate(large: Model, small: Model, x, cond, uncond, cfg_scale, sigmas, eps=1e-8,
                    r_out=None, stream=None):
    """Runs calibration in place on x [B, ...]; returns r [n_steps, B] (device fp32)."""
    import torch
    sig = np.ascontiguousarray(sigmas, dtype=np.float32)
    n = sig.shape[0] - 1
    B = x.shape[0]
    if r_out is None:
        r_out = torch.empty((n, B), dtype=torch.float32, device=x.device)
    _check(lib().track_calibrate(large.handle, small.handle, _ptr(x), B, _ptr(cond), _ptr(uncond),
                                 cfg_scale, sig.ctypes.data, n, eps, _ptr(r_out), _stream(stream)))
    return r_out


def track_sample(large: Model, small: Model, policy, sigmas, x, cond, uncond, cfg_scale, stream=None):
    pol = np.ascontiguousarray(policy, dtype=np.uint8)
    sig = np.ascontiguousarray(sigmas, dtype=np.float32)
    if pol.shape[0] != sig.shape[0] - 1:
        raise ValueError("policy needs one entry per step")
    _check(lib().track_sample(large.handle, small.handle, pol.ctypes.data, sig.ctypes.data,
                              pol.shape[0], _ptr(x), x.shape[0], _ptr(cond), _ptr(uncond),
                              cfg_scale, _stream(stream)))
    return x


def track_band_disagreement(v_L, v_S, eps=1e-8, out=None, stream=None):
    """Sec. 4.4 band split of Eq. 4 for device fp32 [B, C, F, H, W] tensors -> [B, 6]
    (spatial low/mid/high, temporal low/mid/high)."""
    import torch
    B, C, F, H, W = v_L.shape
    if out is None:
        out = torch.empty((B, 6), dtype=torch.float32, device=v_L.device)
    _check(lib().track_band_disagreement(_ptr(v_L), _ptr(v_S), B, C, F, H, W, eps, _ptr(out),
                                         _stream(stream)))
    return out


def track_multistep_step(x, v, state, sigmas, i, stream=None):
    """Step i of the history-carrying scheduler on device fp32 tensors; state has 2 * x.numel()."""
    sig = np.ascontiguousarray(sigmas, dtype=np.float32)
    n = x.numel()
    if state.numel() != 2 * n or v.numel() != n:
        raise ValueError("state must hold 2 * n floats and v n floats")
    _check(lib().track_multistep_step(_ptr(x), _ptr(v), _ptr(state), n, sig.ctypes.data,
                                      sig.shape[0] - 1, int(i), _stream(stream)))
    return x


def track_sample_multistep(large: Model, small: Model, policy, sigmas, x, cond, uncond, cfg_scale,
                           state=None, stream=None):
    """Eq. 3 over the multistep scheduler; returns (x, state)."""
    import torch
    pol = np.ascontiguousarray(policy, dtype=np.uint8)
    sig = np.ascontiguousarray(sigmas, dtype=np.float32)
    if pol.shape[0] != sig.shape[0] - 1:
        raise ValueError("policy needs one entry per step")
    if state is None:
        state = torch.empty((2,) + tuple(x.shape), dtype=torch.float32, device=x.device)
    _check(lib().track_sample_multistep(large.handle, small.handle, pol.ctypes.data,
                                        sig.ctypes.data, pol.shape[0], _ptr(x), x.shape[0],
                                        _ptr(cond), _ptr(uncond), cfg_scale, _ptr(state),
                                        _stream(stream)))
    return x, state


def track_sample_graph(large: Model, small: Model, policy, sigmas, x, cond, uncond, cfg_scale,
                       stream=None):
    """track_sample replayed from a recorded CUDA graph (first call eager, second records)."""
    pol = np.ascontiguousarray(policy, dtype=np.uint8)
    sig = np.ascontiguousarray(sigmas, dtype=np.float32)
    if pol.shape[0] != sig.shape[0] - 1:
        raise ValueError("policy needs one entry per step")
    _check(lib().track_sample_graph(large.handle, small.handle, pol.ctypes.data, sig.ctypes.data,
                                    pol.shape[0], _ptr(x), x.shape[0], _ptr(cond), _ptr(uncond),
                                    cfg_scale, _stream(stream)))
    return x


# ---------------------------------------------------------------- building blocks
def track_linear(dtype, X, W, bias, epilogue, out, gate=None, stream=None):
    M, K = X.shape
    N = W.shape[0]
    _check(lib().track_linear(int(dtype), _ptr(X), _ptr(W), _ptr(bias), M, N, K, epilogue,
                              _ptr(gate), _ptr(out), out.shape[1], _stream(stream)))
    return out


def track_attention(dtype, Q, K, V, O, stream=None):
    S, H, Lq, hd = Q.shape
    Lk = K.shape[2]
    _check(lib().track_attention(int(dtype), _ptr(Q), _ptr(K), _ptr(V), S, H, Lq, Lk, hd, _ptr(O),
                                 _stream(stream)))
    return O
