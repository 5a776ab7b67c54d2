"""The seeded input generator shared by the oracle and the CUDA path."""
import os

import numpy as np
import pytest

import synth

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def test_splitmix64_reference_vector():
    vals = [int(l) for l in open(os.path.join(GOLDEN, "splitmix64_seed1234567.txt"))
            if l.strip() and not l.startswith("#")]
    s, out = 1234567, []
    for _ in range(5):
        s = (s + synth.GAMMA) & synth.MASK64
        out.append(synth.mix64_int(s))
    assert out == vals


def test_counter_form_equals_sequential_stream():
    state = synth.stream_state(5, 9)
    seq, s = [], state
    for _ in range(40):
        s = (s + synth.GAMMA) & synth.MASK64
        z = synth.mix64_int(s)
        seq.append(2 * sum((z >> (16 * l)) & 0xFFFF for l in range(4)) - 262140)
    assert synth.centred_lane_sums(5, 9, 0, 40).tolist() == seq
    assert synth.centred_lane_sums(5, 9, 17, 23).tolist() == seq[17:]


def test_draw_is_chunk_independent_and_scaled(monkeypatch):
    a = synth.draw(3, 4, (1000,), 0.5)
    monkeypatch.setattr(synth, "_CHUNK", 97)
    assert np.array_equal(synth.draw(3, 4, (1000,), 0.5), a)
    n = synth.centred_lane_sums(3, 4, 0, 1000).astype(np.float32)
    assert np.array_equal(a, n * synth.scale_f32(0.5))
    g = synth.draw(3, 4, (1000,), 0.5, offset=1.0)
    assert np.array_equal(g, (n * synth.scale_f32(0.5)) + np.float32(1.0))


def test_draw_moments():
    a = synth.draw(1, 2, (1 << 20,), 2.0).astype(np.float64)
    assert abs(a.mean()) < 0.01 and abs(a.std() - 2.0) < 0.01
    assert np.max(np.abs(a)) <= 2.0 * np.sqrt(3.0) * 2 + 1e-6      # Irwin-Hall(4) support


def test_weight_specs_layout():
    arch = synth.WORKLOADS["tiny"].large
    specs = synth.weight_specs(arch)
    assert len(specs) == 12 + 27 * arch.layers + 3
    assert [s.tensor_id for s in specs] == list(range(len(specs)))
    by = {s.name: s for s in specs}
    assert by["pe.W"].shape == (256, 64) and by["head.W"].shape == (64, 256)
    assert by["blk3.ffn.W1"].shape == (1024, 256) and by["mod.W"].shape == (1536, 256)
    assert by["txt.W1"].shape == (256, 256) and by["blk0.mod_bias"].shape == (6, 256)
    with pytest.raises(ValueError):
        synth.stream_state(2 ** 32, 0)
