"""The denoiser f_m(x_t, t, c) of Eq. 1, written out plainly in fp64.

Test infrastructure only (see the package docstring).

The paper treats each denoiser as a black box (Sec. 3.1: the pair shares the
latent, output shape, conditioning interface and prediction target, while
"internal architectures and parameter counts may differ").  The denoiser used
here is a Wan-2.1-style video DiT; its definition, fixed by this library, is:

* patchify: latent [C, F, H, W] -> tokens (f, h', w') in row-major order, each
  a vector ordered (c, pf, ph, pw) of length C*pf*ph*pw; patch 1x2x2.
* patch embedding  x0 = tokens @ pe.W^T + pe.b.
* time embedding: 256-wide sinusoid of t (cos half then sin half, frequencies
  10000^(-i/128)), MLP  e = tim.W2 @ SiLU(tim.W1 @ emb + tim.b1) + tim.b2,
  modulation  e0 = mod.W @ SiLU(e) + mod.b  reshaped to [6, d].
* text projection  c = txt.W2 @ GELU_tanh(txt.W1 @ ctx + txt.b1) + txt.b2.
* per block, (shift1, scale1, gate1, shift2, scale2, gate2) = e0 + mod_bias:
  - h = LN(x)*(1+scale1)+shift1; q = RMSNorm_d(h Wq^T + bq)*qn.g,
    k = RMSNorm_d(h Wk^T + bk)*kn.g, v = h Wv^T + bv; heads of hd; 3D RoPE on
    q and k; x += gate1 * (softmax(q k^T / sqrt(hd)) v  Wo^T + bo)
  - h = LN(x)*ln3.g + ln3.b; q = RMSNorm_d(h Wcq^T + b)*cqn.g,
    k = RMSNorm_d(c Wck^T + b)*ckn.g, v = c Wcv^T + b (no RoPE);
    x += softmax(q k^T / sqrt(hd)) v  Wco^T + bco
  - h = LN(x)*(1+scale2)+shift2; x += gate2 * (GELU_tanh(h W1^T + b1) W2^T + b2)
* head: (shift, scale) = e + head_bias; out = (LN(x)*(1+scale)+shift) head.W^T + head.b,
  then unpatchify (exact inverse of patchify).

LN is LayerNorm without affine parameters over d (biased variance, eps 1e-6);
RMSNorm_d is over the full model width d (all heads together, eps 1e-6).
Weights are stored [out, in].
"""
from __future__ import annotations

import math

import numpy as np

# ---------------------------------------------------------------------------
# Precision helper
# ---------------------------------------------------------------------------


def round_bf16(a) -> np.ndarray:
    """Round fp32 values to the nearest bf16 value (ties to even), returned as fp32."""
    a = np.ascontiguousarray(np.asarray(a, dtype=np.float32))
    u = a.view(np.uint32).astype(np.uint64)
    lsb = (u >> np.uint64(16)) & np.uint64(1)
    u = (u + np.uint64(0x7FFF) + lsb) & np.uint64(0xFFFF0000)
    return u.astype(np.uint32).view(np.float32).reshape(a.shape)


# ---------------------------------------------------------------------------
# Primitives
# ---------------------------------------------------------------------------


def linear(x, W, b=None):
    """y = x W^T + b with W stored [out, in]."""
    y = np.asarray(x, dtype=np.float64) @ np.asarray(W, dtype=np.float64).T
    if b is not None:
        y = y + np.asarray(b, dtype=np.float64)
    return y


def layer_norm(x, eps=1e-6):
    """LayerNorm over the last axis without affine parameters, biased variance."""
    x = np.asarray(x, dtype=np.float64)
    mu = x.mean(axis=-1, keepdims=True)
    var = ((x - mu) ** 2).mean(axis=-1, keepdims=True)
    return (x - mu) / np.sqrt(var + eps)


def rms_norm(x, g, eps=1e-6):
    """RMSNorm over the last axis: x / sqrt(mean(x^2) + eps) * g."""
    x = np.asarray(x, dtype=np.float64)
    ms = (x * x).mean(axis=-1, keepdims=True)
    return x / np.sqrt(ms + eps) * np.asarray(g, dtype=np.float64)


def gelu_tanh(u):
    """GELU with the tanh approximation of Hendrycks and Gimpel (2016)."""
    u = np.asarray(u, dtype=np.float64)
    return 0.5 * u * (1.0 + np.tanh(math.sqrt(2.0 / math.pi) * (u + 0.044715 * u ** 3)))


def silu(u):
    """SiLU(u) = u * sigmoid(u)."""
    u = np.asarray(u, dtype=np.float64)
    return u / (1.0 + np.exp(-u))


def sinusoid(t, dim=256):
    """Timestep embedding: [cos(t f_i) for i < dim/2] + [sin(t f_i)], f_i = 10000^(-i/(dim/2))."""
    half = dim // 2
    f = np.power(10000.0, -np.arange(half, dtype=np.float64) / half)
    a = float(t) * f
    return np.concatenate([np.cos(a), np.sin(a)])


def softmax(s):
    """Row softmax over the last axis with the row maximum subtracted."""
    s = np.asarray(s, dtype=np.float64)
    e = np.exp(s - s.max(axis=-1, keepdims=True))
    return e / e.sum(axis=-1, keepdims=True)


def attention(q, k, v):
    """softmax(q k^T / sqrt(hd)) v for q [Lq, hd], k [Lk, hd], v [Lk, hd] (no mask)."""
    q = np.asarray(q, dtype=np.float64)
    k = np.asarray(k, dtype=np.float64)
    v = np.asarray(v, dtype=np.float64)
    p = softmax(q @ k.T / math.sqrt(q.shape[-1]))
    return p @ v


def patchify(x, patch=(1, 2, 2)):
    """[C, F, H, W] -> [L, C*pf*ph*pw], tokens (f, h', w') row-major, vectors ordered (c, pf, ph, pw)."""
    x = np.asarray(x)
    C, F, H, W = x.shape
    pf, ph, pw = patch
    y = x.reshape(C, F // pf, pf, H // ph, ph, W // pw, pw)
    y = y.transpose(1, 3, 5, 0, 2, 4, 6)
    return y.reshape((F // pf) * (H // ph) * (W // pw), C * pf * ph * pw)


def unpatchify(tok, shape, patch=(1, 2, 2)):
    """Inverse of ``patchify`` for a latent of shape (C, F, H, W)."""
    C, F, H, W = shape
    pf, ph, pw = patch
    y = np.asarray(tok).reshape(F // pf, H // ph, W // pw, C, pf, ph, pw)
    y = y.transpose(3, 0, 4, 1, 5, 2, 6)
    return y.reshape(C, F, H, W)


def rope_axis_dims(hd):
    """Per-head dims given to the (frame, height, width) axes: hd-4*floor(hd/6), 2*floor(hd/6), 2*floor(hd/6)."""
    s = hd // 6
    return hd - 4 * s, 2 * s, 2 * s


def token_positions(grid):
    """(f, h', w') integer position of every token of an (Fp, Hp, Wp) grid, row-major."""
    Fp, Hp, Wp = grid
    f, h, w = np.meshgrid(np.arange(Fp), np.arange(Hp), np.arange(Wp), indexing="ij")
    return np.stack([f.ravel(), h.ravel(), w.ravel()], axis=1)


def rope(xh, pos):
    """3D rotary embedding of xh [L, heads, hd] at integer positions pos [L, 3].

    The head dims are split into consecutive (frame, height, width) sections of
    ``rope_axis_dims(hd)`` dims; inside a section of D dims the pair
    (2j, 2j+1), read as the complex number x_{2j} + i x_{2j+1}, is multiplied
    by exp(i * p * 10000^(-2j/D)) with p the token's position on that axis.
    """
    xh = np.asarray(xh, dtype=np.float64)
    hd = xh.shape[-1]
    out = xh.copy()
    start = 0
    for axis, D in enumerate(rope_axis_dims(hd)):
        j = np.arange(D // 2, dtype=np.float64)
        freq = np.power(10000.0, -2.0 * j / D)
        ang = pos[:, axis:axis + 1].astype(np.float64) * freq[None, :]      # [L, D/2]
        c, s = np.cos(ang)[:, None, :], np.sin(ang)[:, None, :]
        a = xh[..., start:start + D:2]
        b = xh[..., start + 1:start + D:2]
        out[..., start:start + D:2] = a * c - b * s
        out[..., start + 1:start + D:2] = a * s + b * c
        start += D
    return out


# ---------------------------------------------------------------------------
# The denoiser
# ---------------------------------------------------------------------------

MATRIX_SUFFIXES = (".W", ".W1", ".W2")


class DiT:
    """One denoiser f_m with its weights (canonical names from ``synth.weight_specs``).

    ``precision`` is "fp32" (weights as given) or "bf16" (weight matrices and
    the text conditioning rounded to bf16 first).  Arithmetic is fp64 either way.
    """

    def __init__(self, arch, weights: dict, precision: str = "fp32", name: str = "model"):
        if precision not in ("fp32", "bf16"):
            raise ValueError(precision)
        self.arch = arch
        self.precision = precision
        self.name = name
        self.w = {}
        for k, v in weights.items():
            v = np.asarray(v, dtype=np.float32)
            if precision == "bf16" and k.endswith(MATRIX_SUFFIXES):
                v = round_bf16(v)
            self.w[k] = v
        self.grid = (arch.frames // arch.patch[0], arch.height // arch.patch[1],
                     arch.width // arch.patch[2])
        self.pos = token_positions(self.grid)

    # -- pieces ------------------------------------------------------------
    def W(self, name):
        return self.w[name].astype(np.float64)

    def time_embedding(self, t):
        """(e [d], e0 [6, d]) for model timestep t."""
        emb = sinusoid(t, self.arch.freq_dim)
        e = linear(silu(linear(emb, self.W("tim.W1"), self.W("tim.b1"))),
                   self.W("tim.W2"), self.W("tim.b2"))
        e0 = linear(silu(e), self.W("mod.W"), self.W("mod.b"))
        return e, e0.reshape(6, self.arch.dim)

    def text_projection(self, ctx):
        ctx = np.asarray(ctx, dtype=np.float32)
        if self.precision == "bf16":
            ctx = round_bf16(ctx)
        h = gelu_tanh(linear(ctx, self.W("txt.W1"), self.W("txt.b1")))
        return linear(h, self.W("txt.W2"), self.W("txt.b2"))

    def heads(self, y):
        L = y.shape[0]
        return y.reshape(L, self.arch.heads, self.arch.head_dim)

    def self_attention(self, i, h, rows=None):
        """Self-attention output of the query tokens ``rows`` (all tokens if None); keys
        and values always come from every token of h."""
        p, eps = f"blk{i}.", self.arch.eps
        rows = np.arange(h.shape[0]) if rows is None else np.asarray(rows)
        q = rms_norm(linear(h[rows], self.W(p + "q.W"), self.W(p + "q.b")), self.W(p + "qn.g"), eps)
        k = rms_norm(linear(h, self.W(p + "k.W"), self.W(p + "k.b")), self.W(p + "kn.g"), eps)
        v = linear(h, self.W(p + "v.W"), self.W(p + "v.b"))
        qh = rope(self.heads(q), self.pos[rows])
        kh, vh = rope(self.heads(k), self.pos), self.heads(v)
        o = np.empty_like(qh)
        for hh in range(self.arch.heads):
            o[:, hh, :] = attention(qh[:, hh, :], kh[:, hh, :], vh[:, hh, :])
        return linear(o.reshape(len(rows), -1), self.W(p + "o.W"), self.W(p + "o.b"))

    def cross_attention(self, i, h, c):
        p, eps = f"blk{i}.", self.arch.eps
        q = rms_norm(linear(h, self.W(p + "cq.W"), self.W(p + "cq.b")), self.W(p + "cqn.g"), eps)
        k = rms_norm(linear(c, self.W(p + "ck.W"), self.W(p + "ck.b")), self.W(p + "ckn.g"), eps)
        v = linear(c, self.W(p + "cv.W"), self.W(p + "cv.b"))
        qh, kh, vh = self.heads(q), self.heads(k), self.heads(v)
        o = np.empty_like(qh)
        for hh in range(self.arch.heads):
            o[:, hh, :] = attention(qh[:, hh, :], kh[:, hh, :], vh[:, hh, :])
        return linear(o.reshape(h.shape[0], -1), self.W(p + "co.W"), self.W(p + "co.b"))

    def ffn(self, i, h):
        p = f"blk{i}."
        u = gelu_tanh(linear(h, self.W(p + "ffn.W1"), self.W(p + "ffn.b1")))
        return linear(u, self.W(p + "ffn.W2"), self.W(p + "ffn.b2"))

    def block(self, i, x, e0, c, rows=None):
        """One transformer block on the residual stream x [L, d]; with ``rows``, the
        block's output at those tokens only (self-attention is the one step that
        mixes tokens, and it reads every token's keys and values)."""
        eps = self.arch.eps
        mod = e0 + self.W(f"blk{i}.mod_bias")
        shift1, scale1, gate1, shift2, scale2, gate2 = mod
        h = layer_norm(x, eps) * (1.0 + scale1) + shift1
        if rows is not None:
            x = x[np.asarray(rows)]
        x = x + gate1 * self.self_attention(i, h, rows)
        h = layer_norm(x, eps) * self.W(f"blk{i}.ln3.g") + self.W(f"blk{i}.ln3.b")
        x = x + self.cross_attention(i, h, c)
        h = layer_norm(x, eps) * (1.0 + scale2) + shift2
        x = x + gate2 * self.ffn(i, h)
        return x

    def embed(self, x):
        tok = patchify(np.asarray(x, dtype=np.float64), self.arch.patch)
        return linear(tok, self.W("pe.W"), self.W("pe.b"))

    def head_tokens(self, x, e):
        """The head's per-token output [L, C*pf*ph*pw] (patchified prediction)."""
        hb = self.W("head_bias")
        shift, scale = e + hb[0], e + hb[1]
        h = layer_norm(x, self.arch.eps) * (1.0 + scale) + shift
        return linear(h, self.W("head.W"), self.W("head.b"))

    def head(self, x, e):
        return unpatchify(self.head_tokens(x, e), self.arch.latent_shape, self.arch.patch)

    # -- whole forward -------------------------------------------------------
    def forward(self, x, t, ctx):
        """f_m(x_t, t, c): latent [C, F, H, W] -> prediction of the same shape (fp64)."""
        e, e0 = self.time_embedding(t)
        c = self.text_projection(ctx)
        h = self.embed(x)
        for i in range(self.arch.layers):
            h = self.block(i, h, e0, c)
        return self.head(h, e)

    def forward_at_tokens(self, x, t, ctx, rows):
        """Rows ``rows`` of patchify(f_m(x_t, t, c)): [len(rows), C*pf*ph*pw].

        Every block but the last runs on all tokens; the last block, whose
        self-attention still reads all tokens' keys and values, and the head
        (per token) run only at ``rows``.  Equal to the same rows of forward()."""
        e, e0 = self.time_embedding(t)
        c = self.text_projection(ctx)
        h = self.embed(x)
        last = self.arch.layers - 1
        for i in range(last):
            h = self.block(i, h, e0, c)
        h = self.block(last, h, e0, c, rows)
        return self.head_tokens(h, e)
