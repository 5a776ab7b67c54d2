"""Host-side logic of bench.py (no GPU): the step walk, score-map provenance."""
import numpy as np
import pytest

import bench
import synth


def test_window_walks_the_trajectory_and_starts_over():
    assert bench.window_steps(50, 5, 20) == list(range(5, 25))
    assert bench.window_steps(4, 3, 6) == [3, 0, 1, 2, 3, 0]
    assert bench.window_steps(8, 0, 0) == []


def test_config_hash_identifies_the_configuration():
    h = {name: bench.config_hash(wl) for name, wl in synth.WORKLOADS.items()}
    assert len(set(h.values())) == len(h)                      # every workload its own
    assert bench.config_hash(synth.WORKLOADS["wan480"]) == h["wan480"]   # stable
    assert all(0 <= v < 2 ** 64 for v in h.values())


def test_host_reader_parses_what_the_library_writes(tmp_path):
    T = pytest.importorskip("paper_2609_30096_gb300")
    try:
        T.lib()
    except OSError as e:        # no CUDA runtime on this host
        pytest.skip(str(e))
    rng = np.random.default_rng(3)
    r = rng.uniform(0.5, 1.5, size=(3, 7)).astype(np.float32)
    path = str(tmp_path / "m.trkscore")
    T.track_score_map_save(path, r, 0x0123456789ABCDEF)
    rr, q, h = bench.read_score_map(path)
    assert h == 0x0123456789ABCDEF
    assert np.array_equal(rr, r)
    assert np.array_equal(q, T.track_mean_score(r))


def test_committed_score_maps_match_their_configuration():
    # A map holds one row per calibration sample for the workload's schedule.  It
    # may hold fewer samples than the workload plans (a shortened calibration,
    # rows are independent and a run resumes by appending); its provenance file
    # then states how many.
    import json
    import os
    for name, wl in synth.WORKLOADS.items():
        path = bench.score_map_path(wl)
        if not os.path.exists(path):
            continue
        r, q, h = bench.read_score_map(path)
        assert h == bench.config_hash(wl), name
        assert r.shape[1] == wl.steps and 1 <= r.shape[0] <= wl.calib_seeds, name
        assert np.all(np.isfinite(r)) and np.all(r >= 0), name
        with open(path[:-len(".trkscore")] + ".json") as f:
            assert json.load(f)["M"] == r.shape[0], name


def test_timed_window_has_the_policys_split():
    rng = np.random.default_rng(0)
    for n, k, count, warm in ((50, 25, 20, 5), (30, 15, 20, 5), (50, 25, 7, 3), (4, 2, 20, 5)):
        for _ in range(5):
            pol = np.zeros(n, np.uint8)
            pol[rng.choice(n, k, replace=False)] = 1
            w = bench.timed_window(pol, warm, count)
            assert warm <= w < warm + n
            got = sum(int(pol[i]) for i in bench.window_steps(n, w, count))
            best = min(abs(sum(int(pol[i]) for i in bench.window_steps(n, v, count))
                           - round(count * k / n)) for v in range(warm, warm + n))
            assert abs(got - round(count * k / n)) == best
    assert bench.timed_window(np.zeros(10, np.uint8), 3, 4) == 3      # all-large: any window


def test_event_timed_classes_carry_their_graph_timed_rate():
    classes = {"gemm": {"ms": 1.0}, "update": {"ms": 0.1, "frac_of_hbm": 0.47},
               "disagreement": {"ms": 0.01, "frac_of_hbm": 0.2}}
    hbm = {"cfg_euler": {"frac_of_hbm": 0.73, "gb_per_s": 4960.0},
           "disagreement": {"frac_of_hbm": 0.34, "gb_per_s": 2300.0},
           "disagreement_update": {"frac_of_hbm": 0.55, "gb_per_s": 3700.0}}
    out = bench.annotate_event_timed(classes, hbm)
    assert out["update"]["graph_timed_frac_of_hbm"] == 0.73
    assert out["disagreement"]["graph_timed_frac_of_hbm"] == 0.55
    assert "graph_timed_frac_of_hbm" not in out["gemm"]
    assert bench.annotate_event_timed({}, hbm) == {}
