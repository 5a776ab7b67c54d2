"""Pins of the oracle's denoiser f_m (the DiT that Eq. 1 treats as a black box).

The paper gives no worked example of a denoiser, so the DiT is pinned by its
components (library routines, closed forms, invariants, brute force) and by
structural tests of the composed block that reduce each branch to a closed
form.  A few planted mistakes (mutants of the oracle) check that the pins bite.
"""
import cmath
import math

import numpy as np
import pytest
import torch
import torch.nn.functional as tF

import synth
from oracle import dit


def T(a):
    return torch.tensor(np.asarray(a), dtype=torch.float64)


# ---------------------------------------------------------------------------
# Primitives
# ---------------------------------------------------------------------------


def test_round_bf16_matches_torch_and_ties_to_even():
    rng = np.random.default_rng(0)
    a = np.concatenate([rng.normal(size=4000).astype(np.float32) * 10.0 ** rng.integers(-6, 6, 4000),
                        np.float32([0.0, -0.0, 1.0, 1 + 2 ** -8, 1 + 3 * 2 ** -8, -(1 + 2 ** -8)])])
    ref = torch.tensor(a).to(torch.bfloat16).to(torch.float32).numpy()
    assert np.array_equal(dit.round_bf16(a), ref)
    assert dit.round_bf16(np.float32([1 + 2 ** -8]))[0] == 1.0                 # tie -> even
    assert dit.round_bf16(np.float32([1 + 3 * 2 ** -8]))[0] == 1 + 2 ** -6     # tie -> even


def test_linear_special_cases_and_brute_force():
    rng = np.random.default_rng(1)
    x = rng.normal(size=(3, 5))
    assert np.allclose(dit.linear(x, np.eye(5)), x)
    W, b = rng.normal(size=(4, 5)), rng.normal(size=4)
    for k in range(5):                                  # one-hot input picks column k of W
        e = np.zeros(5)
        e[k] = 1.0
        assert np.allclose(dit.linear(e, W), W[:, k])
    y = dit.linear(x, W, b)
    for i in range(3):
        for o in range(4):
            s = b[o]
            for k in range(5):
                s += x[i, k] * W[o, k]
            assert y[i, o] == pytest.approx(s, rel=1e-13, abs=1e-13)


def test_layer_norm_and_rms_norm():
    rng = np.random.default_rng(2)
    x = rng.normal(size=(7, 33)) * 3 + 2
    y = dit.layer_norm(x, 1e-6)
    assert np.allclose(y.mean(-1), 0, atol=1e-12)
    assert np.allclose(y.var(-1), 1, atol=1e-5)
    assert np.allclose(y, tF.layer_norm(T(x), (33,), eps=1e-6).numpy(), atol=1e-12)
    assert np.allclose(dit.layer_norm(np.float64([[1, 2, 3]]), 0.0), [[-math.sqrt(1.5), 0, math.sqrt(1.5)]])
    g = rng.normal(size=33)
    z = dit.rms_norm(x, np.ones(33), 1e-6)
    assert np.allclose(np.sqrt((z * z).mean(-1)), 1, atol=1e-6)
    assert np.allclose(dit.rms_norm(x, g, 1e-6), tF.rms_norm(T(x), (33,), T(g), eps=1e-6).numpy(),
                       atol=1e-12)


def test_activations():
    u = np.linspace(-8, 8, 1601)
    assert np.allclose(dit.gelu_tanh(u), tF.gelu(T(u), approximate="tanh").numpy(), atol=1e-14)
    exact = np.array([0.5 * v * (1 + math.erf(v / math.sqrt(2))) for v in u])
    assert np.max(np.abs(dit.gelu_tanh(u) - exact)) < 1e-3           # close to the erf GELU
    assert dit.gelu_tanh(np.float64([0.0]))[0] == 0.0
    assert np.allclose(dit.silu(u), tF.silu(T(u)).numpy(), atol=1e-14)
    assert np.allclose(dit.silu(u) - dit.silu(-u), u, atol=1e-12)    # u*sig(u) + u*sig(-u) = u


def test_sinusoid():
    e0 = dit.sinusoid(0.0, 256)
    assert np.array_equal(e0, np.concatenate([np.ones(128), np.zeros(128)]))
    e = dit.sinusoid(1.0, 256)
    assert e[0] == pytest.approx(math.cos(1.0)) and e[128] == pytest.approx(math.sin(1.0))
    f127 = 10000.0 ** (-127 / 128)
    assert e[127] == pytest.approx(math.cos(f127)) and e[255] == pytest.approx(math.sin(f127))


def test_attention_invariants_and_library():
    rng = np.random.default_rng(3)
    q, k, v = rng.normal(size=(6, 8)), rng.normal(size=(9, 8)), rng.normal(size=(9, 8))
    p = dit.softmax(q @ k.T / math.sqrt(8))
    assert np.allclose(p.sum(-1), 1, atol=1e-14) and np.all(p > 0)
    assert np.allclose(dit.attention(q, k[:1], v[:1]), np.repeat(v[:1], 6, 0))    # one key
    assert np.allclose(dit.attention(np.zeros_like(q), k, v), np.repeat(v.mean(0, keepdims=True), 6, 0))
    perm = rng.permutation(9)
    assert np.allclose(dit.attention(q, k[perm], v[perm]), dit.attention(q, k, v))
    ref = tF.scaled_dot_product_attention(T(q)[None], T(k)[None], T(v)[None])[0].numpy()
    assert np.allclose(dit.attention(q, k, v), ref, atol=1e-13)
    # brute force, one output element
    s = [sum(q[2, d] * k[j, d] for d in range(8)) / math.sqrt(8) for j in range(9)]
    m = max(s)
    w = [math.exp(x - m) for x in s]
    assert dit.attention(q, k, v)[2, 5] == pytest.approx(sum(w[j] * v[j, 5] for j in range(9)) / sum(w))


def test_rope_axis_split():
    assert dit.rope_axis_dims(128) == (44, 42, 42)
    assert dit.rope_axis_dims(64) == (24, 20, 20)


def _rope_by_complex_numbers(xh, pos):
    """Independent restatement with Python complex numbers, element by element."""
    L, H, hd = xh.shape
    out = np.empty_like(xh)
    start = 0
    for axis, D in enumerate(dit.rope_axis_dims(hd)):
        for j in range(D // 2):
            theta = 10000.0 ** (-2.0 * j / D)
            for l in range(L):
                rot = cmath.exp(1j * pos[l, axis] * theta)
                for h in range(H):
                    z = complex(xh[l, h, start + 2 * j], xh[l, h, start + 2 * j + 1]) * rot
                    out[l, h, start + 2 * j], out[l, h, start + 2 * j + 1] = z.real, z.imag
        start += D
    return out


def test_rope_complex_definition_norm_and_relative_position():
    rng = np.random.default_rng(4)
    pos = dit.token_positions((2, 3, 4))
    xh = rng.normal(size=(24, 2, 64))
    y = dit.rope(xh, pos)
    assert np.allclose(y, _rope_by_complex_numbers(xh, pos), atol=1e-12)
    assert np.allclose(np.linalg.norm(y, axis=-1), np.linalg.norm(xh, axis=-1))
    # scores depend on position differences only
    q, k = rng.normal(size=(1, 1, 64)), rng.normal(size=(1, 1, 64))
    pa, pb = np.array([[1, 2, 0]]), np.array([[0, 1, 3]])
    s0 = float(np.sum(dit.rope(q, pa) * dit.rope(k, pb)))
    d = np.array([[3, 5, 7]])
    s1 = float(np.sum(dit.rope(q, pa + d) * dit.rope(k, pb + d)))
    assert s0 == pytest.approx(s1, rel=1e-11)


def test_patchify_roundtrip_counts_and_mapping():
    for name, tokens in (("tiny", 64), ("mid", 3510), ("wan480", 32760), ("wan720", 75600)):
        assert synth.WORKLOADS[name].large.tokens == tokens
    rng = np.random.default_rng(5)
    x = rng.normal(size=(3, 2, 4, 6))
    tok = dit.patchify(x)
    assert tok.shape == (2 * 2 * 3, 12)
    assert np.array_equal(dit.unpatchify(tok, x.shape), x)
    for c in range(3):
        for f in range(2):
            for h in range(4):
                for w in range(6):
                    t = (f * 2 + h // 2) * 3 + w // 2
                    assert tok[t, c * 4 + (h % 2) * 2 + (w % 2)] == x[c, f, h, w]


# ---------------------------------------------------------------------------
# Structural pins of the composed block and of the whole forward
# ---------------------------------------------------------------------------

ARCH = synth.Arch(dim=32, layers=2, heads=2, ffn=64, text_dim=24, text_len=5,
                  frames=2, height=4, width=6)


def _model(arch=ARCH, seed=7, cls=dit.DiT):
    return cls(arch, synth.make_weights(arch, seed))


def _force_mod(m, i, e0, **chunks):
    """Set blk{i}.mod_bias so that chunk values e0 + mod_bias equal the given vectors."""
    idx = dict(shift1=0, scale1=1, gate1=2, shift2=3, scale2=4, gate2=5)
    mb = m.w[f"blk{i}.mod_bias"].astype(np.float64).copy()
    for k, v in chunks.items():
        mb[idx[k]] = v - e0[idx[k]]
    m.w[f"blk{i}.mod_bias"] = mb


def _zero(m, *names):
    for n in names:
        m.w[n] = np.zeros_like(m.w[n])


def _setup(cls=dit.DiT, arch=ARCH):
    m = _model(arch, cls=cls)
    rng = np.random.default_rng(9)
    x = rng.normal(size=(arch.tokens, arch.dim))
    e, e0 = m.time_embedding(np.float32(640.0))
    c = m.text_projection(rng.normal(size=(arch.text_len, arch.text_dim)))
    return m, rng, x, e, e0, c


def check_gates_and_identity(cls=dit.DiT):
    m, rng, x, e, e0, c = _setup(cls)
    _force_mod(m, 0, e0, gate1=np.zeros(32), gate2=np.zeros(32))
    _zero(m, "blk0.co.W", "blk0.co.b")
    return np.allclose(m.block(0, x, e0, c), x, atol=1e-12)


def check_self_attention_branch(cls=dit.DiT):
    # 1 + scale1 = 0 makes every token's input the shift vector s: all value rows
    # equal, so attention returns that row whatever the scores are.
    m, rng, x, e, e0, c = _setup(cls)
    s, g1 = rng.normal(size=32), rng.normal(size=32)
    _force_mod(m, 0, e0, shift1=s, scale1=-np.ones(32), gate1=g1, gate2=np.zeros(32))
    _zero(m, "blk0.co.W", "blk0.co.b")
    u = (s @ m.W("blk0.v.W").T + m.W("blk0.v.b")) @ m.W("blk0.o.W").T + m.W("blk0.o.b")
    return np.allclose(m.block(0, x, e0, c), x + g1 * u, atol=1e-12)


def check_ffn_branch(cls=dit.DiT):
    m, rng, x, e, e0, c = _setup(cls)
    s, g2 = rng.normal(size=32), rng.normal(size=32)
    _force_mod(m, 0, e0, gate1=np.zeros(32), shift2=s, scale2=-np.ones(32), gate2=g2)
    _zero(m, "blk0.co.W", "blk0.co.b")
    hid = s @ m.W("blk0.ffn.W1").T + m.W("blk0.ffn.b1")
    hid = 0.5 * hid * (1 + np.tanh(math.sqrt(2 / math.pi) * (hid + 0.044715 * hid ** 3)))
    u = hid @ m.W("blk0.ffn.W2").T + m.W("blk0.ffn.b2")
    return np.allclose(m.block(0, x, e0, c), x + g2 * u, atol=1e-12)


def check_cross_attention_branch(cls=dit.DiT):
    # one text token: cross-attention returns its value row for every query
    arch = synth.Arch(dim=32, layers=1, heads=2, ffn=64, text_dim=24, text_len=1,
                      frames=2, height=4, width=6)
    m, rng, x, e, e0, c = _setup(cls, arch)
    _force_mod(m, 0, e0, gate1=np.zeros(32), gate2=np.zeros(32))
    u = (c[0] @ m.W("blk0.cv.W").T + m.W("blk0.cv.b")) @ m.W("blk0.co.W").T + m.W("blk0.co.b")
    return np.allclose(m.block(0, x, e0, c), x + u, atol=1e-12)


def check_self_attention_against_torch(cls=dit.DiT):
    # The self-attention branch against torch's rms_norm / complex multiply / sdpa.
    m, rng, x, e, e0, c = _setup(cls)
    h = rng.normal(size=(ARCH.tokens, 32))
    W = lambda n: T(m.W("blk0." + n))
    q = tF.rms_norm(T(h) @ W("q.W").T + W("q.b"), (32,), W("qn.g"), eps=1e-6)
    k = tF.rms_norm(T(h) @ W("k.W").T + W("k.b"), (32,), W("kn.g"), eps=1e-6)
    v = T(h) @ W("v.W").T + W("v.b")
    L, H, hd = ARCH.tokens, 2, 16
    pos = dit.token_positions((2, 2, 3))

    def rot(t):
        t = t.reshape(L, H, hd // 2, 2)
        z = torch.view_as_complex(t.contiguous())
        ang = []
        for axis, D in enumerate(dit.rope_axis_dims(hd)):
            fr = 10000.0 ** (-2.0 * torch.arange(D // 2, dtype=torch.float64) / D)
            ang.append(torch.tensor(pos[:, axis], dtype=torch.float64)[:, None] * fr[None])
        ang = torch.cat(ang, 1)[:, None, :]
        return torch.view_as_real(z * torch.polar(torch.ones_like(ang), ang)).reshape(L, H, hd)

    qh, kh, vh = rot(q), rot(k), v.reshape(L, H, hd)
    o = tF.scaled_dot_product_attention(qh.transpose(0, 1), kh.transpose(0, 1), vh.transpose(0, 1))
    ref = o.transpose(0, 1).reshape(L, 32) @ W("o.W").T + W("o.b")
    return np.allclose(m.self_attention(0, h), ref.numpy(), atol=1e-11)


def check_whole_forward_reduces_to_embed_and_head(cls=dit.DiT):
    # Every block the identity: f(x) = unpatchify(head(embed(x))).
    m = _model(cls=cls)
    rng = np.random.default_rng(10)
    t = np.float32(333.0)
    e, e0 = m.time_embedding(t)
    for i in range(ARCH.layers):
        _force_mod(m, i, e0, gate1=np.zeros(32), gate2=np.zeros(32))
        _zero(m, f"blk{i}.co.W", f"blk{i}.co.b")
    x = rng.normal(size=ARCH.latent_shape)
    ctx = rng.normal(size=(ARCH.text_len, ARCH.text_dim))
    tok = dit.patchify(x) @ m.W("pe.W").T + m.W("pe.b")
    shift, scale = e + m.W("head_bias")[0], e + m.W("head_bias")[1]
    out = (dit.layer_norm(tok) * (1 + scale) + shift) @ m.W("head.W").T + m.W("head.b")
    return np.allclose(m.forward(x, t, ctx), dit.unpatchify(out, ARCH.latent_shape), atol=1e-11)


# Conditioning pins (Eq. 1's t and c enter f_m through these two maps).  The
# architecture is square (frequency, text and model widths all 32) so that
# identity, diagonal and permutation weights are well defined.  Every closed
# form is evaluated element by element with libm's exp and tanh.
SQ = synth.Arch(dim=32, layers=1, heads=2, ffn=64, text_dim=32, text_len=5,
                frames=2, height=4, width=6, freq_dim=32)
_A = np.array([0.5, 1.5, 2.0, -1.0, 0.75, -0.25, 3.0, 1.25] * 4)     # bf16-exact diagonals
_PERM = np.array([(7 * i + 3) % 32 for i in range(32)])              # a permutation of 0..31


def _silu1(u):
    return u / (1.0 + math.exp(-u))


def _gelu1(u):
    return 0.5 * u * (1.0 + math.tanh(math.sqrt(2.0 / math.pi) * (u + 0.044715 * u ** 3)))


def _perm_matrix(p):
    P = np.zeros((len(p), len(p)))
    P[np.arange(len(p)), p] = 1.0                       # (P v)[i] = v[p[i]]
    return P


def check_time_embedding_identity(cls=dit.DiT, precision="fp32"):
    # Identity W1, W2 and stacked identity mod.W, zero biases: e = SiLU(emb) and
    # every one of the six rows of e0 is SiLU(e).
    m = cls(SQ, synth.make_weights(SQ, 3), precision)
    d = SQ.dim
    m.w["tim.W1"], m.w["tim.W2"] = np.eye(d), np.eye(d)
    m.w["mod.W"] = np.tile(np.eye(d), (6, 1))
    _zero(m, "tim.b1", "tim.b2", "mod.b")
    t = np.float32(421.0)
    emb = dit.sinusoid(t, d)
    e, e0 = m.time_embedding(t)
    want_e = np.array([_silu1(v) for v in emb])
    want_row = np.array([_silu1(v) for v in want_e])
    ok = e.shape == (d,) and e0.shape == (6, d) and np.allclose(e, want_e, atol=1e-14)
    return ok and all(np.allclose(e0[k], want_row, atol=1e-14) for k in range(6))


def check_time_embedding_structured(cls=dit.DiT, precision="fp32"):
    # W1 = diag(a), W2 = a permutation P, mod.W = six stacked diagonals diag(c_k),
    # random biases:  e[i] = SiLU(a_p(i) emb_p(i) + b1_p(i)) + b2[i] and
    # e0[k, i] = c_k[i] SiLU(e[i]) + mod.b[k d + i]  (row k of the [6, d] reshape
    # is the k-th block of d outputs).
    m = cls(SQ, synth.make_weights(SQ, 4), precision)
    d = SQ.dim
    rng = np.random.default_rng(21)
    c = dit.round_bf16(rng.choice([0.5, -1.0, 2.0, 1.5, -0.75], size=(6, d)).astype(np.float32))
    m.w["tim.W1"], m.w["tim.W2"] = np.diag(_A), _perm_matrix(_PERM)
    m.w["mod.W"] = np.concatenate([np.diag(c[k]) for k in range(6)])
    b1, b2, mb = rng.normal(size=d), rng.normal(size=d), rng.normal(size=6 * d)
    m.w["tim.b1"], m.w["tim.b2"], m.w["mod.b"] = b1, b2, mb
    t = np.float32(87.0)
    emb = dit.sinusoid(t, d)
    e, e0 = m.time_embedding(t)
    want_e = np.array([_silu1(_A[_PERM[i]] * emb[_PERM[i]] + b1[_PERM[i]]) + b2[i] for i in range(d)])
    want_e0 = np.array([[c[k, i] * _silu1(want_e[i]) + mb[k * d + i] for i in range(d)]
                        for k in range(6)])
    return np.allclose(e, want_e, atol=1e-13) and np.allclose(e0, want_e0, atol=1e-13)


def check_text_projection_structured(cls=dit.DiT, precision="fp32"):
    # W1 = diag(a), W2 = a permutation P, random biases:
    # c[l, i] = GELU_tanh(a_p(i) ctx[l, p(i)] + b1_p(i)) + b2[i], with ctx rounded to
    # bf16 first in bf16 mode (the conditioning is fed to the tensor cores in bf16).
    m = cls(SQ, synth.make_weights(SQ, 5), precision)
    d = SQ.dim
    rng = np.random.default_rng(22)
    m.w["txt.W1"], m.w["txt.W2"] = np.diag(_A), _perm_matrix(_PERM)
    b1, b2 = rng.normal(size=d), rng.normal(size=d)
    m.w["txt.b1"], m.w["txt.b2"] = b1, b2
    ctx = rng.normal(size=(SQ.text_len, d)).astype(np.float32)
    ctx[0, :] = np.float32(1.0 + 2.0 ** -10)            # not bf16-representable: rounds to 1
    cin = dit.round_bf16(ctx) if precision == "bf16" else ctx.astype(np.float64)
    got = m.text_projection(ctx)
    want = np.array([[_gelu1(_A[_PERM[i]] * float(cin[l, _PERM[i]]) + b1[_PERM[i]]) + b2[i]
                      for i in range(d)] for l in range(SQ.text_len)])
    return got.shape == (SQ.text_len, d) and np.allclose(got, want, atol=1e-13)


def check_text_projection_bf16(cls=dit.DiT):
    return check_text_projection_structured(cls, "bf16")


def check_time_embedding_bf16(cls=dit.DiT):
    return check_time_embedding_structured(cls, "bf16")


CHECKS = [check_gates_and_identity, check_self_attention_branch, check_ffn_branch,
          check_cross_attention_branch, check_self_attention_against_torch,
          check_whole_forward_reduces_to_embed_and_head, check_time_embedding_identity,
          check_time_embedding_structured, check_time_embedding_bf16,
          check_text_projection_structured, check_text_projection_bf16]


@pytest.mark.parametrize("layers", [1, 2])
def test_forward_at_tokens_is_rows_of_forward(layers):
    # Only self-attention mixes tokens, so the sampled-token forward must give
    # the same rows as the whole forward, in the order asked, for any depth.
    arch = synth.Arch(dim=32, layers=layers, heads=2, ffn=64, text_dim=24, text_len=5,
                      frames=2, height=4, width=6)
    m = _model(arch)
    rng = np.random.default_rng(layers)
    x = rng.normal(size=arch.latent_shape)
    ctx = rng.normal(size=(arch.text_len, arch.text_dim))
    t = np.float32(433.0)
    full = dit.patchify(m.forward(x, t, ctx), arch.patch)
    for rows in (np.arange(arch.tokens), np.array([arch.tokens - 1, 0, 5, 3]), np.array([7])):
        got = m.forward_at_tokens(x, t, ctx, rows)
        assert got.shape == (len(rows), full.shape[1])
        assert np.allclose(got, full[rows], rtol=1e-12, atol=1e-12)


@pytest.mark.parametrize("check", CHECKS, ids=lambda f: f.__name__)
def test_structural_pin(check):
    assert check()


# Planted mistakes: each mutant of the oracle must fail at least one structural pin.

class SwappedGates(dit.DiT):
    def block(self, i, x, e0, c):
        mod = (e0 + self.W(f"blk{i}.mod_bias"))[[0, 1, 5, 3, 4, 2]]
        return dit.DiT.block(self, i, x, mod - self.W(f"blk{i}.mod_bias"), c)


class ShiftScaleSwapped(dit.DiT):
    def block(self, i, x, e0, c):
        mod = (e0 + self.W(f"blk{i}.mod_bias"))[[1, 0, 2, 4, 3, 5]]
        return dit.DiT.block(self, i, x, mod - self.W(f"blk{i}.mod_bias"), c)


class CrossValuesFromLatent(dit.DiT):
    def cross_attention(self, i, h, c):
        return dit.DiT.cross_attention(self, i, h, h)     # keys/values from the latent tokens


class HeadDropsShift(dit.DiT):
    def head(self, x, e):
        hb = self.W("head_bias")
        h = dit.layer_norm(x, self.arch.eps) * (1.0 + e + hb[1])
        out = dit.linear(h, self.W("head.W"), self.W("head.b"))
        return dit.unpatchify(out, self.arch.latent_shape, self.arch.patch)


class TransposedRope(dit.DiT):
    def self_attention(self, i, h, rows=None):
        saved = dit.rope
        dit.rope = lambda xh, pos: saved(xh, pos[:, ::-1].copy())
        try:
            return dit.DiT.self_attention(self, i, h, rows)
        finally:
            dit.rope = saved


class TimeNoSiluBeforeModulation(dit.DiT):
    def time_embedding(self, t):
        emb = dit.sinusoid(t, self.arch.freq_dim)
        e = dit.linear(dit.silu(dit.linear(emb, self.W("tim.W1"), self.W("tim.b1"))),
                       self.W("tim.W2"), self.W("tim.b2"))
        e0 = dit.linear(e, self.W("mod.W"), self.W("mod.b"))
        return e, e0.reshape(6, self.arch.dim)


class TimeSwappedLayers(dit.DiT):
    def time_embedding(self, t):
        emb = dit.sinusoid(t, self.arch.freq_dim)
        e = dit.linear(dit.silu(dit.linear(emb, self.W("tim.W2"), self.W("tim.b1"))),
                       self.W("tim.W1"), self.W("tim.b2"))
        e0 = dit.linear(dit.silu(e), self.W("mod.W"), self.W("mod.b"))
        return e, e0.reshape(6, self.arch.dim)


class TimeModulationTransposed(dit.DiT):
    def time_embedding(self, t):
        e, e0 = dit.DiT.time_embedding(self, t)
        return e, e0.reshape(-1).reshape(self.arch.dim, 6).T


class TextGeluAfterSecondLayer(dit.DiT):
    def text_projection(self, ctx):
        ctx = np.asarray(ctx, dtype=np.float32)
        if self.precision == "bf16":
            ctx = dit.round_bf16(ctx)
        h = dit.linear(ctx, self.W("txt.W1"), self.W("txt.b1"))
        return dit.gelu_tanh(dit.linear(h, self.W("txt.W2"), self.W("txt.b2")))


class TextSwappedLayers(dit.DiT):
    def text_projection(self, ctx):
        ctx = np.asarray(ctx, dtype=np.float32)
        if self.precision == "bf16":
            ctx = dit.round_bf16(ctx)
        h = dit.gelu_tanh(dit.linear(ctx, self.W("txt.W2"), self.W("txt.b1")))
        return dit.linear(h, self.W("txt.W1"), self.W("txt.b2"))


class TextNoBf16Rounding(dit.DiT):
    def text_projection(self, ctx):
        h = dit.gelu_tanh(dit.linear(np.asarray(ctx, dtype=np.float64), self.W("txt.W1"),
                                     self.W("txt.b1")))
        return dit.linear(h, self.W("txt.W2"), self.W("txt.b2"))


@pytest.mark.parametrize("mutant", [SwappedGates, ShiftScaleSwapped, CrossValuesFromLatent,
                                    HeadDropsShift, TransposedRope, TimeNoSiluBeforeModulation,
                                    TimeSwappedLayers, TimeModulationTransposed,
                                    TextGeluAfterSecondLayer, TextSwappedLayers,
                                    TextNoBf16Rounding], ids=lambda c: c.__name__)
def test_planted_mistakes_are_caught(mutant):
    def passes(check):
        try:
            return bool(check(mutant))
        except ValueError:          # a shape mismatch also exposes the mistake
            return False
    failed = [c.__name__ for c in CHECKS if not passes(c)]
    assert failed
