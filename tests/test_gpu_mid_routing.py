"""Calibration and routed sampling at the mid workload's full width and token count (GPU).

The mid pair (1536- and 768-wide DiTs, 12 and 6 heads, FFN 8960 and 3072, latent
16x9x30x52 = 3510 tokens, text 512x4096, 4 Euler steps with shift 5, no CFG,
K = 2) in bf16 tensor-core mode, with the depth cut to 2 and 1 blocks: every
block runs the same kernels at the same shapes, and the fp64 oracle then takes
seconds per forward instead of a minute.  (One evaluation of each model at full
depth is compared in test_gpu_track.py.)

Calibration (Sec. 3.2.1, Eq. 4-5) over M = 2 samples and routed sampling (Eq. 3)
with the resulting policy are compared with the oracle: scores within the bound
that the per-step bf16 tolerance implies, the policy from the GPU's scores
identical to the oracle's (the oracle's K-th/(K+1)-th gap exceeds 1e-3, which is
asserted), and the routed sample within the trajectory tolerance.
"""
import dataclasses

import numpy as np
import pytest

import synth
from oracle import dit, track
from test_gpu_track import check_policy_rule, dev, rel_l2, score_bound

torch = pytest.importorskip("torch")
pytestmark = [pytest.mark.gpu, pytest.mark.slow]

MID = synth.WORKLOADS["mid"]
LARGE = dataclasses.replace(MID.large, layers=2)
SMALL = dataclasses.replace(MID.small, layers=1)
M_CALIB = 2


@pytest.fixture(scope="module")
def T():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2609_30096_gb300 import _build
    _build.build()
    import paper_2609_30096_gb300 as T
    return T


@pytest.fixture(scope="module")
def pair(T):
    wL = synth.make_weights(LARGE, synth.SEED_LARGE)
    wS = synth.make_weights(SMALL, synth.SEED_SMALL)
    L = T.track_model_create(LARGE, list(wL.values()), T.BF16)
    S = T.track_model_create(SMALL, list(wS.values()), T.BF16)
    oL = dit.DiT(LARGE, wL, "bf16", name="L")
    oS = dit.DiT(SMALL, wS, "bf16", name="S")
    yield L, S, oL, oS
    L.close()
    S.close()


@pytest.fixture(scope="module")
def oracle_scores(pair):
    _, _, oL, oS = pair
    x, c, _ = synth.calibration_inputs(LARGE, 0, M_CALIB, with_uncond=False)
    sig = track.schedule(MID.steps, MID.shift)
    r, finals = track.calibrate(oL, oS, x, c, None, MID.cfg, sig)
    return x, c, sig, r, finals


def test_mid_shapes_calibration_scores_and_policy(T, pair, oracle_scores, parity_report):
    L, S, _, _ = pair
    x, c, sig, r_ref, finals = oracle_scores
    xd = dev(x)
    r = T.track_calibrate(L, S, xd, dev(c), None, MID.cfg, sig)
    T.track_sync()
    r_gpu = r.cpu().numpy().T                                  # [M, N]
    q_gpu, q_ref = T.track_mean_score(r_gpu), track.mean_score(r_ref)
    dr = np.abs(r_gpu - r_ref)
    dq = np.abs(q_gpu.astype(np.float64) - q_ref)
    gap = check_policy_rule(T, q_gpu, q_ref, MID.k)
    parity_report(precision="bf16", max_abs_dr=float(dr.max()), max_abs_dq=float(dq.max()),
                  oracle_gap_k=gap, K=MID.k, q_oracle=[float(v) for v in q_ref])
    assert np.all(dr <= score_bound("bf16", r_ref)), float(dr.max())
    for j in range(M_CALIB):                                   # the all-large samples
        assert rel_l2(xd[j].cpu().numpy(), finals[j]) < 5e-2


def test_mid_shapes_routed_sample_follows_the_oracle(T, pair, oracle_scores, parity_report):
    L, S, oL, oS = pair
    _, _, sig, r_ref, _ = oracle_scores
    pol = track.topk_policy(track.mean_score(r_ref), MID.k)
    x, c, _ = synth.evaluation_inputs(LARGE, 0, 1, with_uncond=False)
    xd = dev(x)
    T.track_sample(L, S, pol, sig, xd, dev(c), None, MID.cfg)
    T.track_sync()
    cnt = {}
    ref = track.sample_routed(oL, oS, pol, x[0], c[0], None, MID.cfg, sig, counter=cnt)
    err = rel_l2(xd[0].cpu().numpy(), ref)
    parity_report(precision="bf16", routed_rel_l2=err, policy="".join("S" if p else "L" for p in pol))
    assert cnt == {"L": int((pol == 0).sum()), "S": int(pol.sum())}
    assert err < 5e-2
