"""Pins of the oracle's method functions (Eq. 1-7, Sec. 3.2.1, Sec. 3.3) against what the paper fixes.

Each test checks the oracle against something other than itself: closed forms,
invariants, special cases and brute force.  No GPU is needed.
"""
import itertools
import math

import numpy as np
import pytest

import synth
from oracle import dit, track

# ---------------------------------------------------------------------------
# Scheduler grid and update (Eq. 2 instance)
# ---------------------------------------------------------------------------


@pytest.mark.parametrize("n", [1, 2, 4, 8, 30, 50])
@pytest.mark.parametrize("shift", [1.0, 3.0, 5.0])
def test_schedule_endpoints_and_decreasing(n, shift):
    s = track.schedule(n, shift)
    assert s.dtype == np.float32 and s.shape == (n + 1,)
    assert s[0] == 1.0 and s[-1] == 0.0
    assert np.all(np.diff(s.astype(np.float64)) < 0)


def test_schedule_shift_one_is_uniform():
    s = track.schedule(8, 1.0)
    assert np.array_equal(s, np.float32([1, 0.875, 0.75, 0.625, 0.5, 0.375, 0.25, 0.125, 0]))


def test_schedule_shift_scales_the_odds():
    # The shifted grid multiplies the noise odds sigma/(1-sigma) of the uniform grid by s.
    n, s = 10, 5.0
    sig = track.schedule(n, s).astype(np.float64)[1:-1]
    u = 1.0 - np.arange(1, n) / n
    assert np.allclose(sig / (1 - sig), s * u / (1 - u), rtol=1e-6)
    # mid-grid closed form: sigma_hat = 1/2 -> s/(s+1)
    assert abs(float(track.schedule(8, s)[4]) - s / (s + 1)) < 1e-7


def test_euler_constant_field_sums_the_grid():
    # sum of (sigma_{i+1} - sigma_i) over the grid is sigma_N - sigma_0 = -1
    sig = track.schedule(7, 5.0)
    x = np.array([0.3, -1.0, 2.0])
    c = np.array([1.5, -0.25, 4.0])
    for i in range(7):
        x = track.euler_update(x, c, sig[i], sig[i + 1])
    assert np.allclose(x, np.array([0.3, -1.0, 2.0]) - c, atol=1e-12)


def test_euler_integrates_the_straight_path_exactly():
    # x_sigma = (1 - sigma) x0 + sigma eps has constant velocity eps - x0;
    # starting from eps at sigma_0 = 1, Euler lands on x0 at sigma_N = 0.
    rng = np.random.default_rng(0)
    x0, eps = rng.normal(size=50), rng.normal(size=50)
    sig = track.schedule(13, 5.0)
    x = eps.copy()
    for i in range(13):
        x = track.euler_update(x, eps - x0, sig[i], sig[i + 1])
    assert np.allclose(x, x0, atol=1e-12)


# ---------------------------------------------------------------------------
# Guidance (Eq. 1)
# ---------------------------------------------------------------------------


def test_cfg_special_cases():
    rng = np.random.default_rng(1)
    fc, fu = rng.normal(size=20), rng.normal(size=20)
    assert np.array_equal(track.guided(fc, None, 1.0), fc)          # w = 1: uncond not needed
    assert np.array_equal(track.guided(fc, fu * np.nan, 1.0), fc)   # ... and not read
    assert np.allclose(track.guided(fc, fu, 0.0), fu)                # w = 0: unconditional
    assert np.allclose(track.guided(fc, fc, 7.5), fc)                # equal branches
    # affine in w with slope f_c - f_u
    assert np.allclose(track.guided(fc, fu, 3.0) - track.guided(fc, fu, 2.0), fc - fu)


# ---------------------------------------------------------------------------
# Disagreement (Eq. 4) and mean score (Eq. 5)
# ---------------------------------------------------------------------------


def test_disagreement_special_cases():
    rng = np.random.default_rng(2)
    pl = rng.normal(size=(4, 3, 5))
    assert track.disagreement(pl, pl) == 0.0
    assert track.disagreement(pl, np.zeros_like(pl)) == pytest.approx(1.0, abs=1e-15)
    assert track.disagreement(pl, 2 * pl) == pytest.approx(1.0, abs=1e-14)
    assert track.disagreement(pl, -pl) == pytest.approx(2.0, abs=1e-14)
    ps = rng.normal(size=pl.shape)
    r = track.disagreement(pl, ps)
    assert track.disagreement(3.5 * pl, 3.5 * ps) == pytest.approx(r, rel=1e-14)
    assert r >= 0
    # p_L = 0: the denominator is clamped to eps
    assert track.disagreement(np.zeros(6), np.full(6, 0.5), eps=1e-3) == pytest.approx(
        math.sqrt(6 * 0.25) / 1e-3, rel=1e-14)


def test_disagreement_brute_force():
    rng = np.random.default_rng(3)
    pl, ps = rng.normal(size=17), rng.normal(size=17)
    num = 0.0
    den = 0.0
    for a, b in zip(pl.tolist(), ps.tolist()):
        num += (b - a) * (b - a)
        den += a * a
    assert track.disagreement(pl, ps) == pytest.approx(math.sqrt(num) / math.sqrt(den), rel=1e-13)


def test_mean_score_hand_values():
    q = track.mean_score([[1.0, 2.0, 0.5], [3.0, 4.0, 0.25]])
    assert q.dtype == np.float32
    assert np.array_equal(q, np.float32([2.0, 3.0, 0.375]))


# ---------------------------------------------------------------------------
# Policy (Eq. 6-7 and top-K)
# ---------------------------------------------------------------------------


@pytest.mark.parametrize("seed", range(6))
def test_topk_matches_brute_force(seed):
    rng = np.random.default_rng(seed)
    n = int(rng.integers(1, 11))
    q = rng.uniform(0, 1, size=n).astype(np.float32)
    if seed % 2:                      # many ties
        q = np.round(q * 3).astype(np.float32) / 3
    for k in range(n + 1):
        assert np.array_equal(track.topk_policy(q, k), track.brute_force_topk(q, k)), (q, k)


@pytest.mark.parametrize("seed", range(4))
def test_topk_equals_threshold_solution(seed):
    # Choosing C0 strictly between the K-th and (K+1)-th smallest W = q^2 makes the
    # threshold solution of Eq. 7 select exactly the top-K set, and it is optimal for Eq. 6.
    rng = np.random.default_rng(100 + seed)
    n = 12
    q = rng.uniform(0, 1, size=n).astype(np.float32)
    w = np.sort(q.astype(np.float64) ** 2)
    for k in range(1, n):
        c0 = 0.5 * (w[k - 1] + w[k])
        pol = track.topk_policy(q, k)
        assert np.array_equal(track.threshold_policy(q, c0), pol)
        best = track.relaxed_objective(pol, q, c0)
        for combo in itertools.combinations(range(n), k):
            beta = np.zeros(n)
            beta[list(combo)] = 1
            assert track.relaxed_objective(beta, q, c0) >= best - 1e-15


def test_topk_extremes_and_errors():
    q = np.float32([0.3, 0.1, 0.2])
    assert np.array_equal(track.topk_policy(q, 0), [0, 0, 0])
    assert np.array_equal(track.topk_policy(q, 3), [1, 1, 1])
    assert np.array_equal(track.topk_policy(q, 1), [0, 1, 0])
    assert np.array_equal(track.topk_policy(np.float32([0.5, 0.5, 0.5]), 2), [1, 1, 0])
    for bad_k in (-1, 4):
        with pytest.raises(ValueError):
            track.topk_policy(q, bad_k)
    with pytest.raises(ValueError):
        track.topk_policy(np.float32([0.1, np.nan]), 1)
    with pytest.raises(ValueError):
        track.topk_policy(np.float32([0.1, -0.2]), 1)


def test_topk_on_paper_shaped_score_maps():
    n, k = 50, 25
    i = np.arange(n)
    # U-shaped map with its minimum in the latter half (Sec. 4.4, Fig. 3): a contiguous middle block
    u = (0.6 * ((i - 31) / 31.0) ** 2 + 0.05).astype(np.float32)
    sel = np.flatnonzero(track.topk_policy(u, k))
    assert np.all(np.diff(sel) == 1) and sel[0] > 0 and sel[-1] < n - 1
    assert sel.mean() > n / 2 - 1
    # monotone decreasing map (distilled pipelines, App. B): the last K steps
    m = np.linspace(1.0, 0.1, n).astype(np.float32)
    assert np.array_equal(track.topk_policy(m, k), track.last_k_policy(n, k))


# ---------------------------------------------------------------------------
# Calibration and routed sampling with a tiny denoiser pair
# ---------------------------------------------------------------------------

ARCH_L = synth.Arch(dim=32, layers=2, heads=2, ffn=64, text_dim=24, text_len=5,
                    frames=2, height=4, width=6)
ARCH_S = synth.Arch(dim=16, layers=1, heads=1, ffn=32, text_dim=24, text_len=5,
                    frames=2, height=4, width=6)


@pytest.fixture(scope="module")
def pair():
    L = dit.DiT(ARCH_L, synth.make_weights(ARCH_L, 11), name="L")
    S = dit.DiT(ARCH_S, synth.make_weights(ARCH_S, 12), name="S")
    return L, S


@pytest.fixture(scope="module")
def samples():
    return synth.calibration_inputs(ARCH_L, 0, 2, with_uncond=True)


def test_calibration_follows_the_all_large_trajectory(pair, samples):
    # Sec. 3.2.1: the large model's prediction advances the trajectory, so the
    # calibration latents are those of all-large sampling, bit for bit.
    L, S = pair
    x, c, u = samples
    sig = track.schedule(4, 5.0)
    r, finals = track.calibrate(L, S, x, c, u, 5.0, sig)
    assert r.shape == (2, 4) and np.all(r > 0)
    for j in range(2):
        ref = track.sample_routed(L, S, np.zeros(4, np.uint8), x[j], c[j], u[j], 5.0, sig)
        assert np.array_equal(finals[j], ref)


def test_identical_pair_has_zero_disagreement(samples):
    L = dit.DiT(ARCH_L, synth.make_weights(ARCH_L, 11), name="L")
    S = dit.DiT(ARCH_L, synth.make_weights(ARCH_L, 11), name="S")
    x, c, u = samples
    r, _ = track.calibrate(L, S, x, c, u, 5.0, track.schedule(3, 5.0))
    assert np.all(r == 0.0)


def test_routed_sampling_extremes_and_one_model_per_step(pair, samples):
    L, S = pair
    x, c, u = samples
    sig = track.schedule(5, 5.0)
    all_l = track.sample_routed(L, S, np.zeros(5, np.uint8), x[0], c[0], u[0], 5.0, sig)
    assert np.array_equal(track.sample_routed(L, S, track.topk_policy(np.ones(5, np.float32), 0),
                                              x[0], c[0], u[0], 5.0, sig), all_l)
    all_s = track.sample_routed(L, S, np.ones(5, np.uint8), x[0], c[0], u[0], 5.0, sig)
    ref_s = track.sample_routed(S, L, np.zeros(5, np.uint8), x[0], c[0], u[0], 5.0, sig)
    assert np.array_equal(all_s, ref_s)
    pol = np.uint8([0, 1, 1, 0, 1])
    cnt = {}
    track.sample_routed(L, S, pol, x[0], c[0], u[0], 5.0, sig, counter=cnt)
    assert cnt == {"L": 2 * 2, "S": 3 * 2}     # cond + uncond of exactly one model per step
    cnt = {}
    track.sample_routed(L, S, pol, x[0], c[0], None, 1.0, sig, counter=cnt)
    assert cnt == {"L": 2, "S": 3}             # w = 1: no unconditional pass


def test_mutation_flipped_disagreement_ratio_is_caught():
    # A plausible slip (normalising by the small model's norm) fails the p_S = 0 pin.
    def wrong(pl, ps, eps=1e-8):
        pl, ps = np.ravel(pl), np.ravel(ps)
        return math.sqrt(np.dot(ps - pl, ps - pl)) / max(math.sqrt(np.dot(ps, ps)), eps)
    pl = np.ones(4)
    assert track.disagreement(pl, np.zeros(4)) == pytest.approx(1.0)
    assert wrong(pl, np.zeros(4)) != pytest.approx(1.0)


def test_equal_budget_policies():
    for n in (1, 4, 7, 50):
        for k in range(n + 1):
            f, l = track.first_k_policy(n, k), track.last_k_policy(n, k)
            assert f.sum() == k and l.sum() == k
            assert np.all(f[:k] == 1) and np.all(l[n - k:] == 1)
            r = track.random_k_policy(n, k, seed=123)
            assert r.sum() == k and set(np.unique(r)) <= {0, 1}
    # every step is chosen with probability K/N (uniform subsets)
    n, k = 10, 3
    counts = np.zeros(n)
    for seed in range(4000):
        counts += track.random_k_policy(n, k, seed)
    assert np.allclose(counts / 4000, k / n, atol=0.03)


# ---------------------------------------------------------------------------
# Multistep scheduler with history h_i (Eq. 2), routed (Sec. 3.1)
# ---------------------------------------------------------------------------


def _drive(update, field, sig, x0):
    """Runs a scheduler update over the grid with v_i = field(x_i, sigma_i)."""
    x, state = np.asarray(x0, np.float64), None
    for i in range(len(sig) - 1):
        x, state = update(i, x, field(x, float(sig[i])), state, sig)
    return x


@pytest.mark.parametrize("n,shift", [(2, 5.0), (4, 5.0), (7, 3.0), (50, 5.0)])
def test_multistep_integrates_sigma_linear_fields_exactly(n, shift):
    # For v = a + b*sigma the ODE integral is x_0 + a*(s_N - s_0) + b*(s_N^2 - s_0^2)/2:
    # the trapezoid corrector and the linear-extrapolation predictor are both exact
    # for a linear integrand, on the shifted (non-uniform) grid.  Euler is not.
    rng = np.random.default_rng(n)
    a, b, x0 = rng.normal(size=(3, 17))
    sig = track.schedule(n, shift)
    s0, sN = float(sig[0]), float(sig[-1])
    exact = x0 + a * (sN - s0) + b * (sN * sN - s0 * s0) / 2
    got = _drive(track.multistep_update, lambda x, s: a + b * s, sig, x0)
    assert np.allclose(got, exact, rtol=0, atol=1e-12)
    if n > 1:
        euler = _drive(lambda i, x, p, st, sg: (track.euler_update(x, p, sg[i], sg[i + 1]), None),
                       lambda x, s: a + b * s, sig, x0)
        assert np.max(np.abs(euler - exact)) > 1e-3


def test_multistep_is_second_order():
    # dx/dsigma = lam * x from sigma = 1 to 0: x_N = x_0 * exp(-lam).  The global
    # error falls 4x per halving of the step (the model is evaluated at the
    # predicted latent, as the scheme prescribes); Euler's falls 2x.
    lam, x0 = 1.3, np.array([0.7, -1.1])
    exact = x0 * math.exp(-lam)
    def err(upd, n):
        return np.max(np.abs(_drive(upd, lambda x, s: lam * x, track.schedule(n, 1.0), x0) - exact))
    e = [err(track.multistep_update, n) for n in (64, 128, 256)]
    assert 3.6 < e[0] / e[1] < 4.4 and 3.6 < e[1] / e[2] < 4.4
    eu = lambda i, x, p, st, sg: (track.euler_update(x, p, sg[i], sg[i + 1]), None)
    assert 1.8 < err(eu, 64) / err(eu, 128) < 2.2


def test_multistep_single_step_and_constant_field():
    rng = np.random.default_rng(3)
    x0, c = rng.normal(size=(2, 5))
    sig = track.schedule(1, 5.0)
    one = _drive(track.multistep_update, lambda x, s: c, sig, x0)
    assert np.array_equal(one, track.euler_update(x0, c, sig[0], sig[1]))   # no history yet
    for n in (3, 9):
        got = _drive(track.multistep_update, lambda x, s: c, track.schedule(n, 5.0), x0)
        assert np.allclose(got, x0 - c, rtol=0, atol=1e-14)                 # sum of steps = -1


def test_multistep_history_survives_model_switches(samples):
    # Two distinct model objects computing the same function: any routing must give
    # the single-model trajectory, which fails if a switch touched the history.
    L = dit.DiT(ARCH_L, synth.make_weights(ARCH_L, 11), name="L")
    S = dit.DiT(ARCH_L, synth.make_weights(ARCH_L, 11), name="S")
    x, c, u = samples
    sig = track.schedule(5, 5.0)
    ref = track.sample_routed_multistep(L, S, np.zeros(5, np.uint8), x[0], c[0], u[0], 5.0, sig)
    cnt = {}
    got = track.sample_routed_multistep(L, S, np.uint8([0, 1, 1, 0, 1]), x[0], c[0], u[0], 5.0,
                                        sig, counter=cnt)
    assert np.array_equal(got, ref)
    assert cnt == {"L": 2 * 2, "S": 3 * 2}     # still exactly one model per step


def test_multistep_mutants_are_caught(samples):
    # Plausible slips each fail one of the pins above.
    L = dit.DiT(ARCH_L, synth.make_weights(ARCH_L, 11), name="L")
    S = dit.DiT(ARCH_L, synth.make_weights(ARCH_L, 11), name="S")
    x, c, u = samples
    sig = track.schedule(5, 5.0)
    # (1) history reset whenever the model changes
    def reset_on_switch(pol):
        xx, st, prev = np.asarray(x[0], np.float64), None, None
        for i in range(5):
            m = S if pol[i] else L
            if prev is not None and m is not prev:
                st = None
            p = track.guided_prediction(m, xx, sig[i], c[0], u[0], 5.0)
            if st is None and i > 0:   # restart: Euler from here, as a fresh scheduler would
                xx, st = xx + (float(sig[i + 1]) - float(sig[i])) * p, (xx, p)
            else:
                xx, st = track.multistep_update(i, xx, p, st, sig)
            prev = m
        return xx
    ref = track.sample_routed_multistep(L, S, np.zeros(5, np.uint8), x[0], c[0], u[0], 5.0, sig)
    assert not np.array_equal(reset_on_switch(np.uint8([0, 1, 1, 0, 1])), ref)
    # (2) step ratio inverted, (3) corrector dropped: the sigma-linear pin fails
    rng = np.random.default_rng(0)
    a, b, x0 = rng.normal(size=(3, 9))
    g = track.schedule(6, 5.0)
    exact = x0 + a * (float(g[-1]) - float(g[0])) + b * (float(g[-1]) ** 2 - float(g[0]) ** 2) / 2
    def inverted(i, xx, p, st, sg):
        if st is None:
            return xx + (float(sg[i + 1]) - float(sg[i])) * p, (xx, p)
        xc_prev, v_prev = st
        hp, h = float(sg[i]) - float(sg[i - 1]), float(sg[i + 1]) - float(sg[i])
        xc = xc_prev + 0.5 * hp * (v_prev + p)
        r = hp / h
        return xc + h * ((1 + r / 2) * p - (r / 2) * v_prev), (xc, p)
    def no_corrector(i, xx, p, st, sg):
        if st is None:
            return xx + (float(sg[i + 1]) - float(sg[i])) * p, (xx, p)
        _, v_prev = st
        hp, h = float(sg[i]) - float(sg[i - 1]), float(sg[i + 1]) - float(sg[i])
        r = h / hp
        return xx + h * ((1 + r / 2) * p - (r / 2) * v_prev), (xx, p)
    for wrong in (inverted, no_corrector):
        assert np.max(np.abs(_drive(wrong, lambda xx, s: a + b * s, g, x0) - exact)) > 1e-4


# ---------------------------------------------------------------------------
# Frequency-band decomposition of the disagreement (Sec. 4.4)
# ---------------------------------------------------------------------------


@pytest.mark.parametrize("shape", [(1, 1, 1, 1), (2, 3, 4, 5), (16, 9, 30, 52), (3, 4, 6, 8)])
def test_band_disagreement_parseval(shape):
    # The transform is orthonormal, so each band triple's squares add up to r^2 of Eq. 4.
    rng = np.random.default_rng(sum(shape))
    pl, ps = rng.normal(size=(2,) + shape)
    b = track.band_disagreement(pl, ps)
    r = track.disagreement(pl, ps)
    assert b.shape == (6,) and np.all(b >= 0)
    assert abs(float(np.sum(b[:3] ** 2)) - r * r) < 1e-12 * r * r
    assert abs(float(np.sum(b[3:] ** 2)) - r * r) < 1e-12 * r * r


def test_band_disagreement_brute_force_dft():
    # A direct triple-loop DFT with the bands decided in floating point (no bin of
    # this shape sits on a band edge) gives the same numbers.
    rng = np.random.default_rng(7)
    C, F, H, W = 2, 3, 4, 7
    pl, ps = rng.normal(size=(2, C, F, H, W))
    d = ps - pl
    e_sp, e_t = np.zeros(3), np.zeros(3)
    ff, hh, ww = np.meshgrid(np.arange(F), np.arange(H), np.arange(W), indexing="ij")
    for c in range(C):
        for kf in range(F):
            for kh in range(H):
                for kw in range(W):
                    ph = np.exp(-2j * np.pi * (kf * ff / F + kh * hh / H + kw * ww / W))
                    e = abs(np.sum(d[c] * ph)) ** 2 / (F * H * W)
                    nf, nh, nw = (min(k, n - k) / n for k, n in ((kf, F), (kh, H), (kw, W)))
                    rho_s, rho_t = math.hypot(nh, nw) / 0.5, nf / 0.5
                    e_sp[0 if rho_s < 1 / 3 else 1 if rho_s < 2 / 3 else 2] += e
                    e_t[0 if rho_t < 1 / 3 else 1 if rho_t < 2 / 3 else 2] += e
    ref = np.sqrt(np.concatenate([e_sp, e_t])) / np.linalg.norm(pl)
    assert np.allclose(track.band_disagreement(pl, ps), ref, rtol=1e-12, atol=0)


@pytest.mark.parametrize("k,band", [(2, 0), (12, 1), (24, 2)])
def test_band_disagreement_spatial_tone(k, band):
    # A difference that is a pure horizontal tone of k cycles over W = 52 (radius
    # 2k/52 of Nyquist) puts all its energy in that spatial band and, being
    # constant over frames, in the low temporal band.
    C, F, H, W = 2, 9, 30, 52
    pl = np.ones((C, F, H, W))
    tone = np.cos(2 * np.pi * k * np.arange(W) / W)
    ps = pl + np.broadcast_to(tone, (C, F, H, W))
    b = track.band_disagreement(pl, ps)
    r = track.disagreement(pl, ps)
    assert abs(b[band] - r) < 1e-12 * r and abs(b[3] - r) < 1e-12 * r
    assert np.sum(np.delete(b[:3], band) ** 2) < 1e-24 * r * r


@pytest.mark.parametrize("k,band", [(1, 0), (2, 1), (4, 2)])
def test_band_disagreement_temporal_tone(k, band):
    C, F, H, W = 1, 9, 6, 8
    pl = np.ones((C, F, H, W))
    tone = np.cos(2 * np.pi * k * np.arange(F) / F)[None, :, None, None]
    ps = pl + np.broadcast_to(tone, (C, F, H, W))
    b = track.band_disagreement(pl, ps)
    r = track.disagreement(pl, ps)
    assert abs(b[3 + band] - r) < 1e-12 * r and abs(b[0] - r) < 1e-12 * r


def test_band_disagreement_special_cases_and_edges():
    rng = np.random.default_rng(1)
    pl = rng.normal(size=(3, 4, 6, 8))
    assert np.all(track.band_disagreement(pl, pl) == 0.0)
    b = track.band_disagreement(pl, pl + 0.5)            # a constant offset is all DC
    assert b[1] == b[2] == b[4] == b[5] == 0.0 or max(b[1], b[2], b[4], b[5]) < 1e-12 * b[0]
    # edges: exactly 1/3 of Nyquist belongs to mid, exactly 2/3 to high
    assert track.spatial_band(0, 1, 4, 6) == 1          # |kw|/W = 1/6 -> rho = 1/3
    assert track.spatial_band(0, 2, 4, 6) == 2          # rho = 2/3
    assert track.temporal_band(1, 6) == 1 and track.temporal_band(2, 6) == 2
    assert track.temporal_band(5, 6) == 1               # bin 5 of 6 is frequency -1
