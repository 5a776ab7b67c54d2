"""Seeded synthetic inputs for TRACK workloads (weights, latents, text conditioning).

This module is the one piece of code that both the CUDA path (through its
Python binding, the benchmark and the tests) and the CPU oracle use: it holds
shapes, seeds and a counter-based random generator, and none of the method's
arithmetic.  The paper releases no weights, prompts or latents, so every input
is drawn here from a fixed recipe:

* generator: the i-th output of a SplitMix64 stream (Steele, Lea and Flood,
  "Fast splittable pseudorandom number generators", OOPSLA 2014; the mixing
  constants are those of that generator's public reference implementation)
  whose initial state is ``mix64(seed * 2**32 + tensor_id)``.  Output ``i`` of
  the stream is ``mix64(state + (i + 1) * GAMMA)``, so any element can be
  drawn on its own (counter-based), on the host or on the device.
* approximately normal draws: the four 16-bit lanes of one 64-bit output are
  summed (an Irwin-Hall sum of four uniforms), centred to an even integer
  ``n`` in [-262140, 262140] and scaled by one fp32 multiply
  ``float(n) * c`` with ``c = float32(sigma * sqrt(3) / 131072)``.  That is
  zero-mean with standard deviation ``sigma`` (to 1e-10 relative), and it is
  bit-exact on any IEEE machine because ``n`` is an exact fp32 integer and the
  product is one correctly rounded multiply.  The CUDA library implements the
  same definition for on-device weight generation; the two are checked equal
  bit for bit by the GPU tests.

Weight recipe (per tensor kind): matrices ``N(0, 1/fan_in)``; biases and
modulation biases ``N(0, 0.02^2)``; norm gains ``1 + N(0, 0.05^2)``; LayerNorm
offsets ``N(0, 0.05^2)``.  Latents ``x_T`` and text conditioning are
``N(0, 1)``.  Seeds: large-model weights 1000, small-model weights 2000;
calibration sample ``j`` uses latent seed ``10000 + j``, conditioning
``20000 + j`` and negative conditioning ``30000 + j``; evaluation and benchmark
sample ``j`` uses ``50000 + j``, ``60000 + j`` and ``70000 + j``.
"""
from __future__ import annotations

import math
from dataclasses import dataclass, field, replace

import numpy as np

MASK64 = (1 << 64) - 1
GAMMA = 0x9E3779B97F4A7C15
_M1 = 0xBF58476D1CE4E5B9
_M2 = 0x94D049BB133111EB
_CHUNK = 1 << 22

SEED_LARGE = 1000
SEED_SMALL = 2000
SEED_LATENT = 10000
SEED_COND = 20000
SEED_UNCOND = 30000
SEED_EVAL = 50000


def mix64_int(z: int) -> int:
    """SplitMix64 output mixing on a Python int (used to derive stream states)."""
    z &= MASK64
    z = ((z ^ (z >> 30)) * _M1) & MASK64
    z = ((z ^ (z >> 27)) * _M2) & MASK64
    return z ^ (z >> 31)


def stream_state(seed: int, tensor_id: int) -> int:
    """Initial state of the stream for (seed, tensor_id)."""
    if not (0 <= seed < 2**32 and 0 <= tensor_id < 2**32):
        raise ValueError("seed and tensor_id must fit in 32 bits")
    return mix64_int((seed << 32) | tensor_id)


def _mix64_np(z: np.ndarray) -> np.ndarray:
    z = (z ^ (z >> np.uint64(30))) * np.uint64(_M1)
    z = (z ^ (z >> np.uint64(27))) * np.uint64(_M2)
    return z ^ (z >> np.uint64(31))


def scale_f32(sigma: float) -> np.float32:
    """fp32 multiplier that maps the centred lane sum to standard deviation sigma."""
    return np.float32(float(sigma) * math.sqrt(3.0) / 131072.0)


def centred_lane_sums(seed: int, tensor_id: int, start: int, count: int) -> np.ndarray:
    """Even integers n_i = 2*(sum of the four 16-bit lanes) - 262140, i in [start, start+count)."""
    state = np.uint64(stream_state(seed, tensor_id))
    idx = np.arange(start + 1, start + count + 1, dtype=np.uint64)
    with np.errstate(over="ignore"):
        z = _mix64_np(state + idx * np.uint64(GAMMA))
    m = np.uint64(0xFFFF)
    s = (z & m) + ((z >> np.uint64(16)) & m) + ((z >> np.uint64(32)) & m) + (z >> np.uint64(48))
    return (s.astype(np.int64) * 2 - 262140).astype(np.int32)


def draw(seed: int, tensor_id: int, shape, sigma: float, offset: float | None = None) -> np.ndarray:
    """fp32 array of approximately N(offset, sigma^2) values, bit-exact across machines.

    ``offset`` (if given) is added with one fp32 add after the fp32 multiply.
    """
    shape = tuple(int(s) for s in shape)
    n = int(np.prod(shape, dtype=np.int64)) if shape else 1
    out = np.empty(n, dtype=np.float32)
    c = scale_f32(sigma)
    for s in range(0, n, _CHUNK):
        e = min(n, s + _CHUNK)
        v = centred_lane_sums(seed, tensor_id, s, e - s).astype(np.float32) * c
        if offset is not None:
            v = v + np.float32(offset)
        out[s:e] = v
    return out.reshape(shape)


# --------------------------------------------------------------------------
# Architectures and workloads
# --------------------------------------------------------------------------

@dataclass(frozen=True)
class Arch:
    """One DiT denoiser: model width, depth and the latent/text shapes it reads."""

    dim: int
    layers: int
    heads: int
    ffn: int
    text_dim: int
    text_len: int
    frames: int
    height: int
    width: int
    in_ch: int = 16
    patch: tuple = (1, 2, 2)
    freq_dim: int = 256
    eps: float = 1e-6

    @property
    def head_dim(self) -> int:
        return self.dim // self.heads

    @property
    def tokens(self) -> int:
        pf, ph, pw = self.patch
        return (self.frames // pf) * (self.height // ph) * (self.width // pw)

    @property
    def patch_len(self) -> int:
        pf, ph, pw = self.patch
        return self.in_ch * pf * ph * pw

    @property
    def latent_shape(self) -> tuple:
        return (self.in_ch, self.frames, self.height, self.width)

    @property
    def latent_numel(self) -> int:
        return self.in_ch * self.frames * self.height * self.width


@dataclass(frozen=True)
class Workload:
    """A large/small pair plus the sampling and calibration settings run on it."""

    name: str
    large: Arch
    small: Arch
    steps: int
    shift: float
    cfg: float
    calib_seeds: int
    k: int
    batch: int = 1
    description: str = ""


def _pair(latent, text, large, small):
    C, F, H, W = latent
    Lt, Dt = text
    mk = lambda d, l, h, f: Arch(dim=d, layers=l, heads=h, ffn=f, text_dim=Dt, text_len=Lt,
                                 frames=F, height=H, width=W, in_ch=C)
    return mk(*large), mk(*small)


_tiny = _pair((16, 4, 8, 8), (32, 256), (256, 4, 4, 1024), (128, 2, 2, 512))
_mid = _pair((16, 9, 30, 52), (512, 4096), (1536, 30, 12, 8960), (768, 12, 6, 3072))
_wan480 = _pair((16, 21, 60, 104), (512, 4096), (5120, 40, 40, 13824), (1536, 30, 12, 8960))
_wan720 = _pair((16, 21, 90, 160), (512, 4096), (5120, 40, 40, 13824), (1536, 30, 12, 8960))

WORKLOADS = {
    "tiny": Workload("tiny", *_tiny, steps=8, shift=5.0, cfg=5.0, calib_seeds=4, k=4,
                     description="tiny pair d256/4L vs d128/2L, latent 16x4x8x8 (64 tokens), "
                                 "text 32x256, 8 Euler steps, shift 5, CFG 5, 4 calibration seeds, K=4"),
    "mid": Workload("mid", *_mid, steps=4, shift=5.0, cfg=1.0, calib_seeds=8, k=2,
                    description="mid pair d1536/30L/12H/FFN8960 vs d768/12L/6H/FFN3072, latent "
                                "16x9x30x52 (3510 tokens), text 512x4096, 4 Euler steps, shift 5, "
                                "no CFG, 8 calibration seeds, K=2"),
    "wan480": Workload("wan480", *_wan480, steps=50, shift=5.0, cfg=5.0, calib_seeds=8, k=25,
                       description="Wan-2.1-shaped 14B/1.3B pair, latent 16x21x60x104 (32760 tokens), "
                                   "text 512x4096, 50 steps, shift 5, CFG 5, 8 seeds, K=25"),
    "wan720": Workload("wan720", *_wan720, steps=4, shift=5.0, cfg=1.0, calib_seeds=8, k=2,
                       description="720p-shaped distilled 14B/1.3B pair, latent 16x21x90x160 "
                                   "(75600 tokens), 4 steps, no CFG, K=2"),
    "serving": Workload("serving", *_wan480, steps=30, shift=5.0, cfg=5.0, calib_seeds=16, k=15,
                        batch=4, description="14B/1.3B pair, 4 x 480p latents, 30 steps, CFG 5 "
                                             "(8 sequences per forward), K=15 from 16 seeds"),
}


# --------------------------------------------------------------------------
# Canonical weight list
# --------------------------------------------------------------------------

GLOBAL_TENSORS = ("pe.W", "pe.b", "txt.W1", "txt.b1", "txt.W2", "txt.b2",
                  "tim.W1", "tim.b1", "tim.W2", "tim.b2", "mod.W", "mod.b")
BLOCK_TENSORS = ("mod_bias", "q.W", "q.b", "k.W", "k.b", "v.W", "v.b", "o.W", "o.b",
                 "qn.g", "kn.g", "ln3.g", "ln3.b",
                 "cq.W", "cq.b", "ck.W", "ck.b", "cv.W", "cv.b", "co.W", "co.b",
                 "cqn.g", "ckn.g", "ffn.W1", "ffn.b1", "ffn.W2", "ffn.b2")
HEAD_TENSORS = ("head_bias", "head.W", "head.b")


@dataclass(frozen=True)
class TensorSpec:
    name: str          # canonical name; block tensors are "blk{i}.{name}"
    shape: tuple
    kind: str          # "W" (matrix), "b" (bias), "g" (norm gain), "beta" (LN offset)
    tensor_id: int

    @property
    def sigma(self) -> float:
        if self.kind == "W":
            return 1.0 / math.sqrt(self.shape[1])
        if self.kind == "b":
            return 0.02
        return 0.05

    @property
    def offset(self):
        return 1.0 if self.kind == "g" else None


def _shape_kind(arch: Arch, name: str):
    d, F, Dt, P = arch.dim, arch.ffn, arch.text_dim, arch.patch_len
    table = {
        "pe.W": ((d, P), "W"), "pe.b": ((d,), "b"),
        "txt.W1": ((d, Dt), "W"), "txt.b1": ((d,), "b"),
        "txt.W2": ((d, d), "W"), "txt.b2": ((d,), "b"),
        "tim.W1": ((d, arch.freq_dim), "W"), "tim.b1": ((d,), "b"),
        "tim.W2": ((d, d), "W"), "tim.b2": ((d,), "b"),
        "mod.W": ((6 * d, d), "W"), "mod.b": ((6 * d,), "b"),
        "mod_bias": ((6, d), "b"),
        "qn.g": ((d,), "g"), "kn.g": ((d,), "g"), "cqn.g": ((d,), "g"), "ckn.g": ((d,), "g"),
        "ln3.g": ((d,), "g"), "ln3.b": ((d,), "beta"),
        "ffn.W1": ((F, d), "W"), "ffn.b1": ((F,), "b"),
        "ffn.W2": ((d, F), "W"), "ffn.b2": ((d,), "b"),
        "head_bias": ((2, d), "b"), "head.W": ((P, d), "W"), "head.b": ((P,), "b"),
    }
    if name in table:
        return table[name]
    proj, part = name.split(".")
    assert proj in ("q", "k", "v", "o", "cq", "ck", "cv", "co"), name
    return ((d, d), "W") if part == "W" else ((d,), "b")


def weight_specs(arch: Arch) -> list:
    """Canonical ordered list of the DiT's tensors; tensor_id is the list index."""
    specs = []
    for n in GLOBAL_TENSORS:
        specs.append((n, n))
    for i in range(arch.layers):
        for n in BLOCK_TENSORS:
            specs.append((f"blk{i}.{n}", n))
    for n in HEAD_TENSORS:
        specs.append((n, n))
    out = []
    for tid, (full, base) in enumerate(specs):
        shape, kind = _shape_kind(arch, base)
        out.append(TensorSpec(full, shape, kind, tid))
    return out


def make_tensor(spec: TensorSpec, seed: int) -> np.ndarray:
    return draw(seed, spec.tensor_id, spec.shape, spec.sigma, spec.offset)


def make_weights(arch: Arch, seed: int) -> dict:
    """All weights of one model as fp32 arrays, keyed by canonical name (ordered)."""
    return {s.name: make_tensor(s, seed) for s in weight_specs(arch)}


def param_count(arch: Arch) -> int:
    return sum(int(np.prod(s.shape)) for s in weight_specs(arch))


def latents(arch: Arch, seeds) -> np.ndarray:
    """x_T for each seed: fp32 [B, C, F, H, W] of N(0, 1) draws."""
    return np.stack([draw(int(s), 0, arch.latent_shape, 1.0) for s in seeds])


def context(arch: Arch, seeds) -> np.ndarray:
    """Text conditioning for each seed: fp32 [B, Lt, Dtxt] of N(0, 1) draws."""
    return np.stack([draw(int(s), 0, (arch.text_len, arch.text_dim), 1.0) for s in seeds])


def calibration_inputs(arch: Arch, first: int, batch: int, with_uncond: bool):
    """(x_T, cond, uncond) of calibration samples first .. first+batch-1 (uncond None if unused)."""
    idx = range(first, first + batch)
    x = latents(arch, [SEED_LATENT + j for j in idx])
    c = context(arch, [SEED_COND + j for j in idx])
    u = context(arch, [SEED_UNCOND + j for j in idx]) if with_uncond else None
    return x, c, u


def evaluation_inputs(arch: Arch, first: int, batch: int, with_uncond: bool):
    """(x_T, cond, uncond) of evaluation samples; disjoint seeds from calibration (50000+)."""
    idx = range(first, first + batch)
    x = latents(arch, [SEED_EVAL + j for j in idx])
    c = context(arch, [SEED_EVAL + 10000 + j for j in idx])
    u = context(arch, [SEED_EVAL + 20000 + j for j in idx]) if with_uncond else None
    return x, c, u
