"""The algorithmic FLOP counts behind the bench's TFLOP/s and roofline figures,
pinned to the operations the oracle's denoiser actually performs.

The oracle's forward is run on small architectures with its matrix products
counted (2 FLOPs per multiply-add of every Linear and of both attention
products); the bench's closed forms must give the same integers.
"""
import numpy as np
import pytest

import bench
import synth
from oracle import dit


class Counter:
    def __init__(self):
        self.linear = 0
        self.attention = 0


@pytest.fixture
def counted(monkeypatch):
    c = Counter()
    linear, attention = dit.linear, dit.attention

    def lin(x, W, b=None):
        x = np.asarray(x)
        rows = 1 if x.ndim == 1 else x.shape[0]
        out, inn = np.asarray(W).shape
        c.linear += 2 * rows * out * inn
        return linear(x, W, b)

    def att(q, k, v):
        Lq, hd = np.asarray(q).shape
        Lk = np.asarray(k).shape[0]
        c.attention += 4 * Lq * Lk * hd
        return attention(q, k, v)

    monkeypatch.setattr(dit, "linear", lin)
    monkeypatch.setattr(dit, "attention", att)
    return c


ARCHS = [
    synth.Arch(dim=64, layers=2, heads=2, ffn=128, text_dim=48, text_len=5, frames=2, height=4,
               width=6),
    synth.Arch(dim=128, layers=1, heads=1, ffn=96, text_dim=32, text_len=7, frames=3, height=2,
               width=4),
]


@pytest.mark.parametrize("arch", ARCHS, ids=["2-block", "1-block"])
def test_forward_flops_match_the_oracles_operations(counted, arch):
    m = dit.DiT(arch, synth.make_weights(arch, 5))
    rng = np.random.default_rng(1)
    x = rng.normal(size=arch.latent_shape)
    ctx = rng.normal(size=(arch.text_len, arch.text_dim))
    m.forward(x, np.float32(321.0), ctx)
    d = arch.dim
    # The time embedding and modulation (matrix-vector products on [d]-sized
    # vectors) are outside the bench's count; everything else is inside it.
    time_mlp = 2 * (arch.freq_dim * d + d * d + d * 6 * d)
    per_request_text = bench.text_flops(arch, 1)
    assert counted.linear + counted.attention == \
        bench.forward_flops(arch, 1) + per_request_text + time_mlp
    # attention alone: self-attention over L tokens and cross-attention to Lt
    L, Lt = arch.tokens, arch.text_len
    assert counted.attention == arch.layers * (4 * L * L * d + 4 * L * Lt * d)


def test_forward_flops_scale_with_sequences():
    a = synth.WORKLOADS["mid"].large
    assert bench.forward_flops(a, 4) == 4 * bench.forward_flops(a, 1)
    assert bench.text_flops(a, 2) == 2 * bench.text_flops(a, 1)
    # the mid large model: 11.38 TFLOP per evaluation of one sequence (text excluded)
    assert abs(bench.forward_flops(a, 1) / 1e12 - 11.381) < 1e-3
