"""The C ABI without a GPU: the library builds and loads, exports every symbol
include/track.h declares, and its host-only entry points (schedule, mean score,
top-K policy, weight layout, argument checks) agree with the oracle."""
import ctypes
import os
import re

import numpy as np
import pytest

import synth
from oracle import track as otrack

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def T():
    from paper_2609_30096_gb300 import _build
    _build.build()
    import paper_2609_30096_gb300 as T
    T.lib()
    return T


def declared_functions():
    src = open(os.path.join(ROOT, "include", "track.h")).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    src = re.sub(r"//[^\n]*", "", src)
    names = set(re.findall(r"\b(track_[a-z0-9_]+)\s*\(", src))
    return sorted(names)


def test_every_declared_symbol_is_exported(T):
    names = declared_functions()
    assert len(names) >= 25
    raw = ctypes.CDLL(T._LIB_PATH)
    missing = [n for n in names if not hasattr(raw, n)]
    assert not missing, missing
    assert T.track_abi_version() == 1


def test_every_declared_symbol_has_a_binding_of_the_same_name(T):
    missing = [n for n in declared_functions() if not callable(getattr(T, n, None))]
    assert not missing, missing


@pytest.mark.parametrize("n,shift", [(1, 5.0), (4, 5.0), (8, 5.0), (50, 5.0), (30, 3.0), (7, 1.0)])
def test_schedule_matches_oracle_bitwise(T, n, shift):
    assert np.array_equal(T.track_schedule(n, shift), otrack.schedule(n, shift))


@pytest.mark.parametrize("seed", range(8))
def test_policy_topk_bit_exact(T, seed):
    rng = np.random.default_rng(seed)
    n = int(rng.integers(1, 60))
    q = rng.uniform(0, 1, n).astype(np.float32)
    if seed % 2:
        q = (np.round(q * 4) / 4).astype(np.float32)        # ties
    for k in sorted({0, n, int(rng.integers(0, n + 1)), n // 2}):
        assert np.array_equal(T.track_policy_topk(q, k), otrack.topk_policy(q, k))
        if n <= 10:
            assert np.array_equal(T.track_policy_topk(q, k), otrack.brute_force_topk(q, k))


def test_policy_topk_rejects_bad_input(T):
    q = np.float32([0.2, 0.1])
    for bad in (dict(q=q, k=-1), dict(q=q, k=3), dict(q=np.float32([0.1, np.nan]), k=1),
                dict(q=np.float32([0.1, -1.0]), k=1)):
        with pytest.raises(T.TrackError) as e:
            T.track_policy_topk(bad["q"], bad["k"])
        assert e.value.code == T.TRACK_EINVAL


def test_mean_score_matches_oracle(T):
    r = np.random.default_rng(3).uniform(0, 2, (16, 50)).astype(np.float32)
    assert np.array_equal(T.track_mean_score(r), otrack.mean_score(r))


@pytest.mark.parametrize("name", ["tiny", "mid", "wan480"])
def test_weight_layout_matches_generator(T, name):
    for arch in (synth.WORKLOADS[name].large, synth.WORKLOADS[name].small):
        specs = synth.weight_specs(arch)
        assert T.track_weight_count(arch) == len(specs)
        for s in specs:
            r, c = T.track_weight_shape(arch, s.tensor_id)
            assert (r, c) == (s.shape if len(s.shape) == 2 else (s.shape[0], 1)), s.name


def test_arch_validation(T):
    a = synth.WORKLOADS["tiny"].large
    bad = synth.Arch(dim=96, layers=1, heads=3, ffn=128, text_dim=64, text_len=4,
                     frames=2, height=4, width=4)       # head_dim 32 unsupported
    with pytest.raises(T.TrackError):
        T.track_weight_count(bad)
    with pytest.raises(T.TrackError):
        T.track_weight_shape(a, 10 ** 6)


def test_equal_budget_policies_bit_exact(T):
    for n in (1, 4, 13, 50):
        for k in sorted({0, 1, n // 2, n}):
            assert np.array_equal(T.track_policy_first_k(n, k), otrack.first_k_policy(n, k))
            assert np.array_equal(T.track_policy_last_k(n, k), otrack.last_k_policy(n, k))
            for seed in (0, 7, 2 ** 40 + 3):
                assert np.array_equal(T.track_policy_random_k(n, k, seed),
                                      otrack.random_k_policy(n, k, seed))
    with pytest.raises(T.TrackError):
        T.track_policy_random_k(4, 5, 1)


def test_gemm_schedule_modes(T):
    for mode in (T.GEMM_DATA_PARALLEL, T.GEMM_STREAM_K, T.GEMM_AUTO):
        T.track_gemm_schedule(mode)
    for bad in (-1, 3, 4, 6, 7, 8):
        with pytest.raises(T.TrackError) as e:
            T.track_gemm_schedule(bad)
        assert e.value.code == T.TRACK_EINVAL


def test_failure_hooks_check_arguments(T):
    # Host-side argument checks only: nothing is launched or allocated here.
    for bad in (-1, 999, 2_000_000_001):
        with pytest.raises(T.TrackError) as e:
            T.track_wait_selftest(bad, stream=0)
        assert e.value.code == T.TRACK_EINVAL
    with pytest.raises(T.TrackError) as e:
        T.track_fail_next_allocations(-1)
    assert e.value.code == T.TRACK_EINVAL
    T.track_fail_next_allocations(0)


def test_gemm_raster_groups(T):
    for group in (1, 8, 32, 65536, 0):
        T.track_gemm_raster(group)
    for bad in (-1, 65537):
        with pytest.raises(T.TrackError) as e:
            T.track_gemm_raster(bad)
        assert e.value.code == T.TRACK_EINVAL


def test_attention_schedule_modes(T):
    for mode in (T.GEMM_DATA_PARALLEL, T.GEMM_STREAM_K, T.GEMM_DATA_PARALLEL | T.ATTN_ONE_TILE,
                 T.GEMM_STREAM_K | T.ATTN_ONE_TILE, T.ATTN_ONE_TILE, T.GEMM_AUTO):
        T.track_attention_schedule(mode)
    for bad in (-1, 3, 7, 8, 12):
        with pytest.raises(T.TrackError) as e:
            T.track_attention_schedule(bad)
        assert e.value.code == T.TRACK_EINVAL


# ---------------------------------------------------------------- score-map file
def test_score_map_round_trip_and_resume(T, tmp_path):
    # The calibration map survives a round trip bit for bit, the stored mean is
    # Eq. 5 of the oracle, and calibrating in two halves (rows are independent
    # samples) then appending gives the same file, mean and policy as all at once.
    rng = np.random.default_rng(3)
    M, N, K = 8, 50, 25
    r = rng.uniform(0.0, 2.0, (M, N)).astype(np.float32)
    whole = tmp_path / "whole.trk"
    T.track_score_map_save(whole, r, config_hash=0xABCDEF0123456789)
    r2, q2, h = T.track_score_map_load(whole)
    assert h == 0xABCDEF0123456789
    assert np.array_equal(r2, r)
    assert np.array_equal(q2, otrack.mean_score(r.astype(np.float64)).astype(np.float32))
    assert np.array_equal(q2, T.track_mean_score(r))
    half = tmp_path / "half.trk"
    T.track_score_map_save(half, r[:3], config_hash=7)
    r_a, _, h_a = T.track_score_map_load(half)
    resumed = tmp_path / "resumed.trk"
    T.track_score_map_save(resumed, np.concatenate([r_a, r[3:]]), config_hash=h_a)
    r3, q3, _ = T.track_score_map_load(resumed)
    assert np.array_equal(r3, r) and np.array_equal(q3, q2)
    assert np.array_equal(T.track_policy_topk(q3, K), otrack.topk_policy(q2, K))


def test_score_map_rejects_bad_files_and_scores(T, tmp_path):
    r = np.ones((2, 4), np.float32)
    good = tmp_path / "good.trk"
    T.track_score_map_save(good, r)
    raw = good.read_bytes()
    assert raw[:8] == b"TRKSCORE" and len(raw) == 28 + 4 * (8 + 4)
    cases = {"truncated": raw[:-3], "magic": b"X" + raw[1:], "version": raw[:8] + b"\x02" + raw[9:],
             "empty": b""}
    for name, data in cases.items():
        p = tmp_path / f"{name}.trk"
        p.write_bytes(data)
        with pytest.raises(T.TrackError) as e:
            T.track_score_map_load(p)
        assert e.value.code == T.TRACK_EINVAL, name
    with pytest.raises(T.TrackError):
        T.track_score_map_load(tmp_path / "missing.trk")
    for bad in (np.float32(-1.0), np.float32(np.nan)):
        rb = r.copy()
        rb[1, 2] = bad
        with pytest.raises(T.TrackError) as e:
            T.track_score_map_save(tmp_path / "bad.trk", rb)
        assert e.value.code == T.TRACK_EINVAL
    with pytest.raises(T.TrackError):
        T.track_score_map_save(tmp_path / "no_such_dir" / "x.trk", r)


def test_disagreement_update_checks_arguments_on_the_host(T):
    # Host-side checks only: every call below is rejected before anything is
    # launched, so the addresses are never dereferenced.
    lib = T.lib()
    n, B = 1024, 2
    base = 1 << 30                                   # stand-in addresses, 16-byte aligned
    vL, vS, acc = base, base + 4 * B * n, base + 8 * B * n
    x_ok = base + 16 * B * n
    cases = [
        (0, vS, B, n, 1e-8, acc, x_ok),              # NULL v_L
        (vL, vS, B, n, 1e-8, acc, 0),                # NULL x
        (vL, vS, B, 0, 1e-8, acc, x_ok),             # empty samples
        (vL, vS, B, n, 0.0, acc, x_ok),              # eps not positive
        (vL, vS, B, n, 1e-8, acc, vL),               # x is v_L
        (vL, vS, B, n, 1e-8, acc, vS + 4 * n),       # x overlaps the second sample of v_S
        (vL, vS, B, n, 1e-8, acc, vL - 4 * n),       # x's second sample overlaps v_L
    ]
    for a, b, bb, nn, eps, ac, x in cases:
        rc = lib.track_disagreement_update(a, b, bb, nn, eps, ac, x, 0.5, 0.25, None)
        assert rc == T.TRACK_EINVAL, (a, b, bb, nn, eps, ac, x)
