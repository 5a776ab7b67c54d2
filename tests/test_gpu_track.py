"""End-to-end parity of the routed denoising hot path against the oracle (GPU).

Tiny pair (fp32 and bf16 modes): per-step guided predictions of both models
(teacher-forced on the oracle's all-large trajectory), calibration scores,
the policy derived from them, routed sampling, and the bit-exact identities
the paper fixes (calibration follows the all-large trajectory; identical
models disagree by exactly zero).  Mid pair (bf16, the benchmark workload at
full size): per-step predictions of both models.
"""
import numpy as np
import pytest

import synth
from oracle import dit, track

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

TOL = {"fp32": 1e-4, "bf16": 2e-2}      # relative L2 of per-step v
SCORE_TOL = 1e-3                         # absolute, per-step disagreement


@pytest.fixture(scope="module")
def T():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2609_30096_gb300 import _build
    _build.build()
    import paper_2609_30096_gb300 as T
    return T


def rel_l2(a, b):
    a = np.asarray(a, np.float64)
    b = np.asarray(b, np.float64)
    return float(np.linalg.norm(a - b) / np.linalg.norm(b))


def dev(a):
    return torch.from_numpy(np.ascontiguousarray(a, dtype=np.float32)).cuda()


WL = synth.WORKLOADS["tiny"]


class Pair:
    def __init__(self, T, prec, wl=WL, small_seed=synth.SEED_SMALL, small_arch=None):
        dtype = T.FP32 if prec == "fp32" else T.BF16
        small_arch = small_arch or wl.small
        wL = synth.make_weights(wl.large, synth.SEED_LARGE)
        wS = synth.make_weights(small_arch, small_seed)
        self.L = T.track_model_create(wl.large, list(wL.values()), dtype)
        self.S = T.track_model_create(small_arch, list(wS.values()), dtype)
        self.oL = dit.DiT(wl.large, wL, prec, name="L")
        self.oS = dit.DiT(small_arch, wS, prec, name="S")


@pytest.fixture(scope="module", params=["fp32", "bf16"])
def tiny(T, request):
    return request.param, Pair(T, request.param)


@pytest.fixture(scope="module")
def calib_inputs():
    return synth.calibration_inputs(WL.large, 0, WL.calib_seeds, with_uncond=True)


@pytest.fixture(scope="module")
def oracle_calibration(tiny, calib_inputs):
    prec, P = tiny
    x, c, u = calib_inputs
    sig = track.schedule(WL.steps, WL.shift)
    # the all-large reference trajectory of every calibration sample, with r
    traj = []
    r = np.zeros((len(x), WL.steps))
    for j in range(len(x)):
        xs = [np.asarray(x[j], np.float64)]
        for k in range(WL.steps):
            pl = track.guided_prediction(P.oL, xs[-1], sig[k], c[j], u[j], WL.cfg)
            ps = track.guided_prediction(P.oS, xs[-1], sig[k], c[j], u[j], WL.cfg)
            r[j, k] = track.disagreement(pl, ps)
            xs.append(track.euler_update(xs[-1], pl, sig[k], sig[k + 1]))
        traj.append(xs)
    return sig, traj, r


def test_per_step_prediction_parity(T, tiny, calib_inputs, oracle_calibration):
    """Teacher-forced: the GPU gets the oracle's x_{t_k}; v of both models within tolerance."""
    prec, P = tiny
    x, c, u = calib_inputs
    sig, traj, _ = oracle_calibration
    cd, ud = dev(c[:2]), dev(u[:2])
    for k in range(WL.steps):
        xk = np.stack([traj[j][k] for j in range(2)]).astype(np.float32)
        t = float(track.model_timestep(sig[k]))
        for gm, om in ((P.L, P.oL), (P.S, P.oS)):
            v = T.track_denoise(gm, dev(xk), t, cd, ud, WL.cfg).cpu().numpy()
            for j in range(2):
                ref = track.guided_prediction(om, xk[j], sig[k], c[j], u[j], WL.cfg)
                err = rel_l2(v[j], ref)
                assert err < TOL[prec], (prec, om.name, k, j, err)


@pytest.mark.parametrize("prec", ["fp32", "bf16"])
@pytest.mark.parametrize("dim,heads", [(2560, 20)])
def test_wide_model_prediction_parity(T, prec, dim, heads):
    """Rows of 2560 features take the block-per-row LayerNorm and RMSNorm/RoPE
    kernels (one block of threads per row, as the 14B shape's 5120 does in the
    full-shape tests); one guided evaluation of a one-block model of that width
    against the oracle."""
    arch = synth.Arch(dim=dim, layers=1, heads=heads, ffn=1024, text_dim=256, text_len=32,
                      frames=2, height=8, width=16)
    w = synth.make_weights(arch, 4242)
    m = T.track_model_create(arch, list(w.values()), T.FP32 if prec == "fp32" else T.BF16)
    x, c, u = synth.evaluation_inputs(arch, 0, 1, with_uncond=True)
    v = T.track_denoise(m, dev(x), 700.0, dev(c), dev(u), 5.0).cpu().numpy()
    m.close()
    ref = track.guided_prediction(dit.DiT(arch, w, prec), x[0], 0.7, c[0], u[0], 5.0)
    assert rel_l2(v[0], ref) < TOL[prec]


def test_no_cfg_prediction_parity(T, tiny, calib_inputs):
    prec, P = tiny
    x, c, _ = calib_inputs
    v = T.track_denoise(P.L, dev(x[:1]), 900.0, dev(c[:1]), None, 1.0).cpu().numpy()
    ref = P.oL.forward(x[0], np.float32(900.0), c[0])
    assert rel_l2(v[0], ref) < TOL[prec]


def score_bound(prec, r_ref):
    """Largest |r_gpu - r_oracle| a calibration score may show.  fp32 mode: the
    score tolerance.  bf16 mode: with p_L and p_S each within relative L2 e of
    the oracle's, r = ||p_S - p_L|| / ||p_L|| moves by at most about
    e (||p_S|| + ||p_L||) / ||p_L|| + e r <= e (2 + 2 r), since ||p_S|| / ||p_L||
    <= 1 + r."""
    if prec == "fp32":
        return SCORE_TOL
    return TOL["bf16"] * (2.0 + 2.0 * np.asarray(r_ref))


def check_policy_rule(T, q_gpu, q_ref, K):
    """The policy from the GPU's scores equals the oracle's wherever the oracle's
    K-th and (K+1)-th lowest scores differ by more than the score tolerance.  The
    workloads' seeds make that gap hold, which is asserted too, so the policy
    comparison always runs."""
    srt = np.sort(np.asarray(q_ref, np.float64))
    gap = float(srt[K] - srt[K - 1])
    assert gap > SCORE_TOL, gap
    assert np.array_equal(T.track_policy_topk(np.asarray(q_gpu, np.float32), K),
                          track.topk_policy(q_ref, K))
    return gap


def test_calibration_scores_and_policy(T, tiny, calib_inputs, oracle_calibration, parity_report):
    prec, P = tiny
    x, c, u = calib_inputs
    sig, traj, r_ref = oracle_calibration
    xd = dev(x)
    r = T.track_calibrate(P.L, P.S, xd, dev(c), dev(u), WL.cfg, sig)
    T.track_sync()
    r_gpu = r.cpu().numpy().T                                  # [M, N]
    dr = np.abs(r_gpu - r_ref)
    q_gpu = T.track_mean_score(r_gpu)
    q_ref = track.mean_score(r_ref)
    dq = np.abs(q_gpu.astype(np.float64) - q_ref)
    gap = check_policy_rule(T, q_gpu, q_ref, WL.k)
    parity_report(precision=prec, max_abs_dr=float(dr.max()), max_abs_dq=float(dq.max()),
                  oracle_gap_k=gap, K=WL.k)
    assert np.all(dr <= score_bound(prec, r_ref)), float(dr.max())
    assert np.max(dq) <= np.max(score_bound(prec, q_ref))
    # the calibration latents end on the oracle's all-large sample
    for j in range(len(x)):
        assert rel_l2(xd[j].cpu().numpy(), traj[j][-1]) < (1e-3 if prec == "fp32" else 5e-2)


def test_calibration_trajectory_is_the_all_large_trajectory(T, tiny, calib_inputs):
    """Sec. 3.2.1: the large model advances the calibration trajectory, so its latents
    equal those of all-large routed sampling bit for bit."""
    prec, P = tiny
    x, c, u = calib_inputs
    sig = track.schedule(WL.steps, WL.shift)
    xa = dev(x)
    T.track_calibrate(P.L, P.S, xa, dev(c), dev(u), WL.cfg, sig)
    xb = dev(x)
    T.track_sample(P.L, P.S, np.zeros(WL.steps, np.uint8), sig, xb, dev(c), dev(u), WL.cfg)
    T.track_sync()
    assert torch.equal(xa, xb)
    xc = dev(x)                                               # K = 0 routed sample
    T.track_sample(P.L, P.S, T.track_policy_topk(np.ones(WL.steps, np.float32), 0), sig, xc,
                   dev(c), dev(u), WL.cfg)
    T.track_sync()
    assert torch.equal(xb, xc)


def test_identical_models_have_zero_disagreement(T, calib_inputs):
    P = Pair(T, "fp32", small_seed=synth.SEED_LARGE, small_arch=WL.large)
    x, c, u = calib_inputs
    r = T.track_calibrate(P.L, P.S, dev(x), dev(c), dev(u), WL.cfg, track.schedule(3, 5.0))
    T.track_sync()
    assert np.all(r.cpu().numpy() == 0.0)


def test_routed_sampling_follows_the_oracle(T, tiny, calib_inputs, oracle_calibration):
    prec, P = tiny
    _, _, r_ref = oracle_calibration
    pol = track.topk_policy(track.mean_score(r_ref), WL.k)
    x, c, u = synth.evaluation_inputs(WL.large, 0, 2, with_uncond=True)
    sig = track.schedule(WL.steps, WL.shift)
    xd = dev(x)
    T.track_sample(P.L, P.S, pol, sig, xd, dev(c), dev(u), WL.cfg)
    T.track_sync()
    cnt = {}
    for j in range(2):
        ref = track.sample_routed(P.oL, P.oS, pol, x[j], c[j], u[j], WL.cfg, sig, counter=cnt)
        assert rel_l2(xd[j].cpu().numpy(), ref) < (1e-3 if prec == "fp32" else 5e-2)
    assert cnt == {"L": 2 * 2 * int((pol == 0).sum()), "S": 2 * 2 * int(pol.sum())}


def test_multistep_routed_sampling_follows_the_oracle(T, tiny, calib_inputs, oracle_calibration):
    prec, P = tiny
    _, _, r_ref = oracle_calibration
    pol = track.topk_policy(track.mean_score(r_ref), WL.k)
    x, c, u = synth.evaluation_inputs(WL.large, 0, 2, with_uncond=True)
    sig = track.schedule(WL.steps, WL.shift)
    xd = dev(x)
    T.track_sample_multistep(P.L, P.S, pol, sig, xd, dev(c), dev(u), WL.cfg)
    T.track_sync()
    for j in range(2):
        ref = track.sample_routed_multistep(P.oL, P.oS, pol, x[j], c[j], u[j], WL.cfg, sig)
        assert rel_l2(xd[j].cpu().numpy(), ref) < (1e-3 if prec == "fp32" else 5e-2)
    # the history is kept across switches: differs from the Euler trajectory
    xe = dev(x)
    T.track_sample(P.L, P.S, pol, sig, xe, dev(c), dev(u), WL.cfg)
    T.track_sync()
    assert not torch.equal(xe, xd)


def test_multistep_identities_bit_exact(T, calib_inputs):
    # Two distinct models with identical weights: any routing reproduces the
    # single-model trajectory bit for bit (a history reset at a switch would not).
    P = Pair(T, "fp32", small_seed=synth.SEED_LARGE, small_arch=WL.large)
    x, c, u = calib_inputs
    sig = track.schedule(WL.steps, WL.shift)
    ref = dev(x[:2])
    T.track_sample_multistep(P.L, P.S, np.zeros(WL.steps, np.uint8), sig, ref, dev(c[:2]),
                             dev(u[:2]), WL.cfg)
    got = dev(x[:2])
    pol = np.array([0, 1, 1, 0, 1, 0, 1, 1][:WL.steps], np.uint8)
    T.track_sample_multistep(P.L, P.S, pol, sig, got, dev(c[:2]), dev(u[:2]), WL.cfg)
    T.track_sync()
    assert torch.equal(got, ref)


def test_graph_replay_matches_eager(T, tiny):
    # First call eager, second records and replays, later calls replay: every
    # call must equal an eager run bit for bit, with the buffers' current
    # contents (new latent values each call, same pointer) and the same kernels.
    prec, P = tiny
    pol = np.array([0, 1, 1, 0, 1, 0, 0, 1][:WL.steps], np.uint8)
    x, c, u = synth.evaluation_inputs(WL.large, 3, 2, with_uncond=True)
    sig = track.schedule(WL.steps, WL.shift)
    s = torch.cuda.Stream()
    with torch.cuda.stream(s):
        cd, ud, xg = dev(c), dev(u), dev(x)
        for call in range(4):
            x_in = torch.from_numpy((x * (1.0 + 0.25 * call)).astype(np.float32)).cuda()
            xg.copy_(x_in)
            n0 = T.track_launch_count()
            T.track_sample_graph(P.L, P.S, pol, sig, xg, cd, ud, WL.cfg, stream=s.cuda_stream)
            n_graph = T.track_launch_count() - n0
            xe = x_in.clone()
            T.track_invalidate_ctx(P.L)
            T.track_invalidate_ctx(P.S)
            n0 = T.track_launch_count()
            T.track_sample(P.L, P.S, pol, sig, xe, cd, ud, WL.cfg, stream=s.cuda_stream)
            n_eager = T.track_launch_count() - n0
            T.track_sync(s.cuda_stream)
            assert torch.equal(xg, xe), call
            assert n_graph == n_eager, call
        # a different policy is a different graph (eager first), still exact
        xg.copy_(dev(x))
        T.track_sample_graph(P.L, P.S, 1 - pol, sig, xg, cd, ud, WL.cfg, stream=s.cuda_stream)
        xe = dev(x)
        T.track_sample(P.L, P.S, 1 - pol, sig, xe, cd, ud, WL.cfg, stream=s.cuda_stream)
        T.track_sync(s.cuda_stream)
        assert torch.equal(xg, xe)
    with pytest.raises(T.TrackError) as e:   # the legacy default stream cannot be recorded
        T.track_sample_graph(P.L, P.S, pol, sig, dev(x), dev(c), dev(u), WL.cfg, stream=0)
    assert e.value.code == T.TRACK_EINVAL


def test_timed_graph_brackets_every_kernel(T, tiny):
    # With kernel timing on, the recorded graph carries the brackets as event
    # nodes: a replay computes the same values and reports the same launches,
    # classes and work as an eager bracketed run, with positive times.
    prec, P = tiny
    pol = np.array([1, 0, 0, 1, 0, 1, 1, 0][:WL.steps], np.uint8)
    x, c, u = synth.evaluation_inputs(WL.large, 5, 1, with_uncond=True)
    sig = track.schedule(WL.steps, WL.shift)
    s = torch.cuda.Stream()
    try:
        with torch.cuda.stream(s):
            cd, ud, xg = dev(c), dev(u), dev(x)
            T.track_profile_enable(True)
            T.track_profile_read()
            xe = dev(x)
            T.track_invalidate_ctx(P.L)
            T.track_invalidate_ctx(P.S)
            T.track_sample(P.L, P.S, pol, sig, xe, cd, ud, WL.cfg, stream=s.cuda_stream)
            T.track_sync(s.cuda_stream)
            eager = T.track_profile_read()
            for call in range(4):   # eager, record + replay, replay, replay
                xg.copy_(dev(x))
                T.track_sample_graph(P.L, P.S, pol, sig, xg, cd, ud, WL.cfg, stream=s.cuda_stream)
                T.track_sync(s.cuda_stream)
                got = T.track_profile_read()
                assert torch.equal(xg, xe), call
                for k in ("gemm", "attention", "cross_attention", "layernorm", "norm_rope",
                          "update"):
                    assert got[k][2] == eager[k][2] > 0, (call, k)
                    assert got[k][1] == eager[k][1], (call, k)
                    assert got[k][0] > 0, (call, k)
    finally:
        T.track_profile_enable(False)
        T.track_profile_read()


def test_abandoned_wait_is_reported_and_the_context_survives(T):
    # The bounded pipeline wait of the tensor-core kernels, made to run out on a
    # barrier nothing completes (about 0.5 ms of SM cycles): the next sync
    # reports the timeout with the self-test's code, clears it, and the device
    # keeps working.
    s = torch.cuda.Stream()
    T.track_sync(s.cuda_stream)
    T.track_wait_selftest(1_000_000, stream=s.cuda_stream)
    with pytest.raises(T.TrackError) as e:
        T.track_sync(s.cuda_stream)
    assert e.value.code == T.TRACK_ETIMEOUT
    assert f"code {T.TRACK_WAIT_SELFTEST_CODE}" in str(e.value)
    T.track_sync(s.cuda_stream)                        # cleared
    X = torch.ones((300, 128), dtype=torch.bfloat16, device="cuda")
    W = torch.eye(128, dtype=torch.bfloat16, device="cuda")
    out = torch.zeros((300, 128), dtype=torch.bfloat16, device="cuda")
    T.track_linear(T.BF16, X, W, None, T.EPI_STORE, out)
    T.track_sync()
    assert torch.equal(out, X)


def test_injected_allocation_failures(T, calib_inputs):
    # A model whose weight allocation fails is not created; a denoise whose
    # workspace allocation fails returns ENOMEM and leaves the model usable.
    x, c, u = calib_inputs
    T.track_fail_next_allocations(1000)
    try:
        with pytest.raises(T.TrackError) as e:
            T.track_model_create_seeded(WL.large, synth.SEED_LARGE, T.BF16)
        assert e.value.code == T.TRACK_ENOMEM
    finally:
        T.track_fail_next_allocations(0)
    m = T.track_model_create_seeded(WL.large, synth.SEED_LARGE, T.BF16)
    T.track_fail_next_allocations(1000)   # every allocation of the call fails
    try:
        with pytest.raises(T.TrackError) as e:
            T.track_denoise(m, dev(x[:1]), 500.0, dev(c[:1]), dev(u[:1]), WL.cfg)
        assert e.value.code == T.TRACK_ENOMEM
    finally:
        T.track_fail_next_allocations(0)
    v1 = T.track_denoise(m, dev(x[:1]), 500.0, dev(c[:1]), dev(u[:1]), WL.cfg)
    v2 = T.track_denoise(m, dev(x[:1]), 500.0, dev(c[:1]), dev(u[:1]), WL.cfg)
    T.track_sync()
    assert torch.equal(v1, v2) and bool(torch.isfinite(v1).all())
    m.close()


def test_argument_errors(T, tiny, calib_inputs):
    prec, P = tiny
    x, c, u = calib_inputs
    with pytest.raises(T.TrackError) as e:
        T.track_denoise(P.L, dev(x[:1]), 500.0, dev(c[:1]), None, 5.0)   # uncond needed
    assert e.value.code == T.TRACK_EINVAL
    other = synth.Arch(dim=128, layers=1, heads=2, ffn=256, text_dim=256, text_len=32,
                       frames=4, height=8, width=16)
    M = T.track_model_create_seeded(other, 5, T.FP32)
    assert not T.track_models_compatible(P.L, M)
    with pytest.raises(T.TrackError):
        T.track_sample(P.L, M, np.zeros(2, np.uint8), track.schedule(2, 5.0), dev(x[:1]),
                       dev(c[:1]), dev(u[:1]), WL.cfg)


# ---------------------------------------------------------------- full-size mid workload
@pytest.mark.slow
@pytest.mark.parametrize("which", ["large", "small"])
def test_mid_workload_full_size_per_step(T, which):
    """The benchmark workload at full size (3510 tokens, 30/12 layers, bf16, no CFG):
    one denoiser evaluation of each model against the fp64 oracle, with weights
    generated on the device exactly as the benchmark creates them."""
    wl = synth.WORKLOADS["mid"]
    arch = getattr(wl, which)
    seed = synth.SEED_LARGE if which == "large" else synth.SEED_SMALL
    m = T.track_model_create_seeded(arch, seed, T.BF16)
    x, c, _ = synth.evaluation_inputs(arch, 0, 1, with_uncond=False)
    sig = track.schedule(wl.steps, wl.shift)
    t = float(track.model_timestep(sig[1]))
    v = T.track_denoise(m, dev(x), t, dev(c), None, 1.0).cpu().numpy()
    m.close()
    ref = dit.DiT(arch, synth.make_weights(arch, seed), "bf16").forward(x[0], np.float32(t), c[0])
    assert rel_l2(v[0], ref) < TOL["bf16"]
