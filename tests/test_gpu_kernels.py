"""Kernel-level parity of the CUDA path against the oracle, through the C ABI.

GEMM (tcgen05 bf16 and FFMA fp32, every epilogue, ragged tiles), attention
(bf16 tensor-core and fp32), guidance / Euler update, the Eq. 4 reduction and
on-device weight generation.
"""
import numpy as np
import pytest

import synth
from oracle import dit, track

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def T():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2609_30096_gb300 import _build
    _build.build()
    import paper_2609_30096_gb300 as T
    return T


DEV = "cuda"


def rel_l2(a, b):
    a = np.asarray(a, np.float64)
    b = np.asarray(b, np.float64)
    return float(np.linalg.norm(a - b) / max(np.linalg.norm(b), 1e-300))


def dev_f32(a):
    return torch.from_numpy(np.ascontiguousarray(a, dtype=np.float32)).to(DEV)


def dev_bf16(a):
    return dev_f32(a).to(torch.bfloat16)


# ---------------------------------------------------------------- GEMM
GEMM_SHAPES = [
    (128, 256, 64),      # one tile
    (200, 384, 128),     # ragged M, N not a multiple of 256 (128-wide tiles)
    (1, 512, 256),       # a single row
    (777, 1024, 640),    # ragged M, several 256-wide tiles, K not a power of two
    (3510, 1536, 1536),  # mid-size output projection (bench shape)
    (600, 8960, 1536),   # wide N (FFN up-projection)
    (333, 1536, 8960),   # long K (FFN down-projection)
]


@pytest.mark.parametrize("M,N,K", GEMM_SHAPES)
@pytest.mark.parametrize("epi", [0, 1, 2, 3])
def test_linear_bf16_tcgen05(T, M, N, K, epi):
    rng = np.random.default_rng(M * 7 + N * 3 + K + epi)
    X = dit.round_bf16(rng.normal(size=(M, K)).astype(np.float32))
    W = dit.round_bf16((rng.normal(size=(N, K)) / np.sqrt(K)).astype(np.float32))
    b = rng.normal(size=N).astype(np.float32) * 0.1
    gate = rng.normal(size=N).astype(np.float32)
    ref = dit.linear(X, W, b)
    if epi == T.EPI_GELU:
        ref = dit.gelu_tanh(ref)
    if epi in (T.EPI_STORE, T.EPI_GELU):
        out = torch.zeros((M, N), dtype=torch.bfloat16, device=DEV)
        T.track_linear(T.BF16, dev_bf16(X), dev_bf16(W), dev_f32(b), epi, out)
        T.track_sync()
        got = out.float().cpu().numpy()
        assert rel_l2(got, ref) < 4e-3
        assert np.all(np.abs(got - ref) <= 8e-3 * np.abs(ref) + 2e-3 * np.sqrt(np.mean(ref ** 2)))
    else:
        r0 = rng.normal(size=(M, N)).astype(np.float32)
        out = dev_f32(r0)
        T.track_linear(T.BF16, dev_bf16(X), dev_bf16(W), dev_f32(b), epi, out,
                       gate=dev_f32(gate) if epi == T.EPI_RESID_GATE else None)
        T.track_sync()
        delta = out.cpu().numpy().astype(np.float64) - r0
        want = ref * gate if epi == T.EPI_RESID_GATE else ref
        assert rel_l2(delta, want) < 2e-5


# Stream-K forced where the shape allows it: a ragged 32-column last tile and
# ragged rows (three CTAs per tile), the output projection at 3510 tokens (two),
# wide N, K = 4096 over 52 tiles, where a tile spans four CTAs, and two shapes of
# several waves, whose leading waves are taken whole before the stream-K tail.
SK_SHAPES = [
    (2000, 1568, 1536),
    (3510, 1536, 1536),
    (600, 8960, 1536),
    (1664, 1024, 4096),
    (8250, 1536, 512),     # 390 tiles: one wave taken whole, the rest stream-K
    (16300, 2048, 256),    # 1024 tiles: five waves whole, ragged rows
]


@pytest.fixture(params=["sk", "dp"])
def schedule(T, request):
    T.track_gemm_schedule({"sk": T.GEMM_STREAM_K, "dp": T.GEMM_DATA_PARALLEL}[request.param])
    yield request.param
    T.track_gemm_schedule(T.GEMM_AUTO)


@pytest.mark.parametrize("M,N,K", SK_SHAPES)
@pytest.mark.parametrize("epi", [0, 1, 2, 3])
def test_linear_bf16_schedules(T, schedule, M, N, K, epi):
    rng = np.random.default_rng(M * 5 + N + K * 3 + epi)
    X = dit.round_bf16(rng.normal(size=(M, K)).astype(np.float32))
    W = dit.round_bf16((rng.normal(size=(N, K)) / np.sqrt(K)).astype(np.float32))
    b = rng.normal(size=N).astype(np.float32) * 0.1
    gate = rng.normal(size=N).astype(np.float32)
    ref = dit.linear(X, W, b)
    if epi == T.EPI_GELU:
        ref = dit.gelu_tanh(ref)
    Xd, Wd, bd = dev_bf16(X), dev_bf16(W), dev_f32(b)
    gd = dev_f32(gate) if epi == T.EPI_RESID_GATE else None
    outs = []
    for _ in range(2):  # twice: same bits (fixed summation order, counters reset)
        if epi in (T.EPI_STORE, T.EPI_GELU):
            out = torch.zeros((M, N), dtype=torch.bfloat16, device=DEV)
        else:
            r0 = rng.normal(size=(M, N)).astype(np.float32) if not outs else r0
            out = dev_f32(r0)
        T.track_linear(T.BF16, Xd, Wd, bd, epi, out, gate=gd)
        T.track_sync()
        outs.append(out.float().cpu().numpy())
    assert np.array_equal(outs[0], outs[1])
    if epi in (T.EPI_STORE, T.EPI_GELU):
        got = outs[0]
        assert rel_l2(got, ref) < 4e-3
        assert np.all(np.abs(got - ref) <= 8e-3 * np.abs(ref) + 2e-3 * np.sqrt(np.mean(ref ** 2)))
    else:
        delta = outs[0].astype(np.float64) - r0
        want = ref * gate if epi == T.EPI_RESID_GATE else ref
        assert rel_l2(delta, want) < 2e-5


def test_linear_bf16_schedules_agree(T):
    # Stream-K differs from data-parallel only in the order of fp32 partial sums.
    rng = np.random.default_rng(11)
    M, N, K = 3510, 1536, 8960
    X = dev_bf16(rng.normal(size=(M, K)).astype(np.float32))
    W = dev_bf16((rng.normal(size=(N, K)) / np.sqrt(K)).astype(np.float32))
    res = []
    for mode in (T.GEMM_DATA_PARALLEL, T.GEMM_STREAM_K):
        T.track_gemm_schedule(mode)
        out = torch.zeros((M, N), dtype=torch.float32, device=DEV)
        T.track_linear(T.BF16, X, W, None, T.EPI_RESID, out)
        T.track_sync()
        res.append(out.cpu().numpy().astype(np.float64))
    T.track_gemm_schedule(T.GEMM_AUTO)
    # Two fp32 sums of K terms in different association differ by about
    # sqrt(K) * 2^-24 relative (6e-6 at K = 8960); the bound allows 3x that.
    assert rel_l2(res[1], res[0]) < 2e-5


@pytest.mark.parametrize("mode", ["dp", "sk"])
def test_linear_bf16_raster_groups_agree(T, mode):
    # The tile order changes which CTA computes a tile, never a data-parallel
    # tile's arithmetic: every raster group gives the same bits (65 row units,
    # ragged).  Under stream-K the order also moves the split points between
    # tiles, so split tiles may round differently (fp32 sums in another order,
    # then bf16): about one bf16 step apart.
    rng = np.random.default_rng(12)
    M, N, K = 8250, 1024, 1536
    X = dev_bf16(rng.normal(size=(M, K)).astype(np.float32))
    W = dev_bf16((rng.normal(size=(N, K)) / np.sqrt(K)).astype(np.float32))
    b = dev_f32(rng.normal(size=N).astype(np.float32))
    T.track_gemm_schedule({"dp": T.GEMM_DATA_PARALLEL, "sk": T.GEMM_STREAM_K}[mode])
    res = []
    try:
        for group in (0, 1, 5, 32, 65536):
            T.track_gemm_raster(group)
            out = torch.zeros((M, N), dtype=torch.bfloat16, device=DEV)
            T.track_linear(T.BF16, X, W, b, T.EPI_STORE, out)
            T.track_sync()
            res.append(out.float().cpu().numpy())
    finally:
        T.track_gemm_raster(0)
        T.track_gemm_schedule(T.GEMM_AUTO)
    for r in res[1:]:
        if mode == "sk":
            scale = np.sqrt(np.mean(res[0] ** 2))
            assert np.all(np.abs(r - res[0]) <= 2.0 ** -7 * np.abs(res[0]) + 1e-3 * scale)
        else:
            assert np.array_equal(r, res[0])
    ref = dit.linear(dit.round_bf16(X.float().cpu().numpy()[::97]), W.float().cpu().numpy(),
                     b.cpu().numpy())
    assert rel_l2(res[0][::97], ref) < 4e-3


@pytest.mark.parametrize("M,N,K", [(1, 32, 64), (100, 96, 80), (513, 700, 256)])
@pytest.mark.parametrize("epi", [0, 1, 2, 3])
def test_linear_fp32(T, M, N, K, epi):
    rng = np.random.default_rng(M + N + K + epi)
    X = rng.normal(size=(M, K)).astype(np.float32)
    W = (rng.normal(size=(N, K)) / np.sqrt(K)).astype(np.float32)
    b = rng.normal(size=N).astype(np.float32)
    gate = rng.normal(size=N).astype(np.float32)
    r0 = rng.normal(size=(M, N)).astype(np.float32)
    out = dev_f32(r0)
    T.track_linear(T.FP32, dev_f32(X), dev_f32(W), dev_f32(b), epi, out,
                   gate=dev_f32(gate) if epi == 2 else None)
    T.track_sync()
    ref = dit.linear(X, W, b)
    if epi == 1:
        ref = dit.gelu_tanh(ref)
    got = out.cpu().numpy().astype(np.float64)
    if epi == 2:
        got, ref = got - r0, ref * gate
    elif epi == 3:
        got = got - r0
    assert rel_l2(got, ref) < 2e-6


def test_linear_rejects_unsupported_bf16_shape(T):
    X = torch.zeros((4, 96), dtype=torch.bfloat16, device=DEV)
    W = torch.zeros((64, 96), dtype=torch.bfloat16, device=DEV)
    out = torch.zeros((4, 64), dtype=torch.bfloat16, device=DEV)
    with pytest.raises(T.TrackError) as e:
        T.track_linear(T.BF16, X, W, None, 0, out)
    assert e.value.code == T.TRACK_EUNSUPPORTED


# ---------------------------------------------------------------- attention
ATTN_CASES = [  # S, H, Lq, Lk, hd
    (1, 1, 64, 64, 64),
    (2, 3, 100, 100, 128),     # ragged query and key tiles
    (1, 2, 257, 32, 64),       # short keys (tiny cross-attention)
    (2, 2, 300, 512, 128),     # cross-attention at text length 512
    (1, 12, 3510, 3510, 128),  # mid-size self-attention (bench shape)
    (4, 16, 1000, 700, 128),   # ragged queries and keys, last key tile under half full
    (2, 40, 600, 512, 64),     # hd 64, text-length keys
]


def _attn_ref(Q, K, V):
    S, H, Lq, hd = Q.shape
    out = np.empty((S, Lq, H, hd))
    for s in range(S):
        for h in range(H):
            out[s, :, h, :] = dit.attention(Q[s, h], K[s, h], V[s, h])
    return out


@pytest.mark.parametrize("S,H,Lq,Lk,hd", ATTN_CASES)
def test_attention_bf16(T, S, H, Lq, Lk, hd):
    rng = np.random.default_rng(Lq + Lk + hd)
    Q = dit.round_bf16(rng.normal(size=(S, H, Lq, hd)).astype(np.float32))
    K = dit.round_bf16(rng.normal(size=(S, H, Lk, hd)).astype(np.float32))
    V = dit.round_bf16(rng.normal(size=(S, H, Lk, hd)).astype(np.float32))
    O = torch.zeros((S, Lq, H, hd), dtype=torch.bfloat16, device=DEV)
    T.track_attention(T.BF16, dev_bf16(Q), dev_bf16(K), dev_bf16(V), O)
    T.track_sync()
    if S * H * Lq * Lk > 20_000_000:  # large case: sampled query rows
        rows = rng.choice(Lq, 64, replace=False)
        ref = _attn_ref(Q[:, :, rows], K, V)
        got = O.float().cpu().numpy()[:, rows]
    else:
        ref, got = _attn_ref(Q, K, V), O.float().cpu().numpy()
    assert rel_l2(got, ref) < 1e-2


@pytest.mark.parametrize("S,H,Lq,Lk,hd", ATTN_CASES[:4])
def test_attention_fp32(T, S, H, Lq, Lk, hd):
    rng = np.random.default_rng(Lq * 3 + Lk + hd)
    Q, K, V = (rng.normal(size=(S, H, L, hd)).astype(np.float32) for L in (Lq, Lk, Lk))
    O = torch.zeros((S, Lq, H, hd), dtype=torch.float32, device=DEV)
    T.track_attention(T.FP32, dev_f32(Q), dev_f32(K), dev_f32(V), O)
    T.track_sync()
    assert rel_l2(O.cpu().numpy(), _attn_ref(Q, K, V)) < 2e-6


@pytest.mark.parametrize("hd", [64, 128])
def test_attention_growing_logits(T, hd):
    # Key norms grow along the sequence and queries are scaled up, so each half
    # of every key tile raises the running row maximum by far more than the
    # lazy-rescaling threshold many times over: every O rescale path runs.
    rng = np.random.default_rng(hd + 7)
    S, H, Lq, Lk = 1, 3, 200, 900
    ramp = (1.0 + 4.0 * np.arange(Lk) / Lk)[None, None, :, None]
    Q = dit.round_bf16((4.0 * rng.normal(size=(S, H, Lq, hd))).astype(np.float32))
    K = dit.round_bf16((ramp * rng.normal(size=(S, H, Lk, hd))).astype(np.float32))
    V = dit.round_bf16(rng.normal(size=(S, H, Lk, hd)).astype(np.float32))
    O = torch.zeros((S, Lq, H, hd), dtype=torch.bfloat16, device=DEV)
    T.track_attention(T.BF16, dev_bf16(Q), dev_bf16(K), dev_bf16(V), O)
    T.track_sync()
    assert rel_l2(O.float().cpu().numpy(), _attn_ref(Q, K, V)) < 1e-2


# Both attention schedules of both kernels (a pair of query tiles per work
# item, and one) at shapes where stream-K splits items over 2 (bench shape,
# ragged keys, hd 64), 3 and 4 CTAs; each run twice for bits.
ATTN_SCHED_CASES = [
    (1, 12, 3510, 3510, 128),
    (4, 16, 1000, 700, 128),
    (1, 4, 2400, 2000, 128),
    (1, 6, 1100, 2000, 128),
    (2, 40, 600, 512, 64),
]


@pytest.fixture(params=["dp", "sk", "one-tile dp", "one-tile sk"])
def attn_schedule(T, request):
    mode = T.GEMM_DATA_PARALLEL if request.param.endswith("dp") else T.GEMM_STREAM_K
    T.track_attention_schedule(mode | (T.ATTN_ONE_TILE if "one-tile" in request.param else 0))
    yield request.param
    T.track_attention_schedule(T.GEMM_AUTO)


@pytest.mark.parametrize("S,H,Lq,Lk,hd", ATTN_SCHED_CASES)
def test_attention_schedules(T, attn_schedule, S, H, Lq, Lk, hd):
    rng = np.random.default_rng(Lq * 5 + Lk + hd + H)
    Q = dit.round_bf16(rng.normal(size=(S, H, Lq, hd)).astype(np.float32))
    K = dit.round_bf16(rng.normal(size=(S, H, Lk, hd)).astype(np.float32))
    V = dit.round_bf16(rng.normal(size=(S, H, Lk, hd)).astype(np.float32))
    Qd, Kd, Vd = dev_bf16(Q), dev_bf16(K), dev_bf16(V)
    outs = []
    for _ in range(2):
        O = torch.zeros((S, Lq, H, hd), dtype=torch.bfloat16, device=DEV)
        T.track_attention(T.BF16, Qd, Kd, Vd, O)
        T.track_sync()
        outs.append(O.float().cpu().numpy())
    assert np.array_equal(outs[0], outs[1])
    rows = rng.choice(Lq, min(Lq, 48), replace=False)
    ref = _attn_ref(Q[:, :, rows], K, V)
    assert rel_l2(outs[0][:, rows], ref) < 1e-2


@pytest.mark.parametrize("hd", [64, 128])
def test_attention_growing_logits_split(T, hd):
    # Stream-K with query tiles split over up to four CTAs whose parts reach
    # very different row maxima: the combine's 2^(m_p - M) weights matter.
    rng = np.random.default_rng(hd + 17)
    S, H, Lq, Lk = 1, 8, 1000, 2000
    ramp = (1.0 + 4.0 * np.arange(Lk) / Lk)[None, None, :, None]
    Q = dit.round_bf16((4.0 * rng.normal(size=(S, H, Lq, hd))).astype(np.float32))
    K = dit.round_bf16((ramp * rng.normal(size=(S, H, Lk, hd))).astype(np.float32))
    V = dit.round_bf16(rng.normal(size=(S, H, Lk, hd)).astype(np.float32))
    T.track_attention_schedule(T.GEMM_STREAM_K)
    try:
        O = torch.zeros((S, Lq, H, hd), dtype=torch.bfloat16, device=DEV)
        T.track_attention(T.BF16, dev_bf16(Q), dev_bf16(K), dev_bf16(V), O)
        T.track_sync()
    finally:
        T.track_attention_schedule(T.GEMM_AUTO)
    rows = rng.choice(Lq, 64, replace=False)
    assert rel_l2(O.float().cpu().numpy()[:, rows], _attn_ref(Q[:, :, rows], K, V)) < 1e-2


def test_attention_single_key_returns_value_row(T):
    rng = np.random.default_rng(5)
    Q = rng.normal(size=(1, 2, 70, 64)).astype(np.float32)
    K = rng.normal(size=(1, 2, 1, 64)).astype(np.float32)
    V = dit.round_bf16(rng.normal(size=(1, 2, 1, 64)).astype(np.float32))
    O = torch.zeros((1, 70, 2, 64), dtype=torch.bfloat16, device=DEV)
    T.track_attention(T.BF16, dev_bf16(Q), dev_bf16(K), dev_bf16(V), O)
    T.track_sync()
    got = O.float().cpu().numpy()
    for h in range(2):
        assert np.array_equal(got[0, :, h, :], np.repeat(V[0, h], 70, 0))


# ---------------------------------------------------------------- frequency bands (Sec. 4.4)
@pytest.mark.parametrize("shape", [(1, 16, 9, 30, 52), (2, 3, 4, 5, 7), (3, 1, 1, 1, 1),
                                   (1, 16, 21, 60, 104)])
def test_band_disagreement_matches_oracle(T, shape):
    rng = np.random.default_rng(sum(shape))
    vl = rng.normal(size=shape).astype(np.float32)
    vs = (vl + 0.3 * rng.normal(size=shape)).astype(np.float32)
    outs = []
    for _ in range(2):
        out = T.track_band_disagreement(dev_f32(vl), dev_f32(vs))
        T.track_sync()
        outs.append(out.cpu().numpy())
    assert np.array_equal(outs[0], outs[1])                     # deterministic
    for b in range(shape[0]):
        ref = track.band_disagreement(vl[b], vs[b])
        assert np.allclose(outs[0][b], ref, rtol=1e-5, atol=1e-6 * np.max(ref))


def test_band_disagreement_tones(T):
    C, F, H, W = 2, 9, 30, 52
    vl = np.ones((3, C, F, H, W), np.float32)
    vs = vl.copy()
    vs[0] += np.cos(2 * np.pi * 12 * np.arange(W) / W).astype(np.float32)         # spatial mid
    vs[1] += np.cos(2 * np.pi * 4 * np.arange(F) / F).astype(np.float32)[:, None, None]  # temporal high
    vs[2] += 0.25                                                                   # DC only
    out = T.track_band_disagreement(dev_f32(vl), dev_f32(vs)).cpu().numpy()
    r = [track.disagreement(vl[b], vs[b]) for b in range(3)]
    assert abs(out[0, 1] - r[0]) < 1e-5 * r[0] and max(out[0, 0], out[0, 2]) < 1e-3 * r[0]
    assert abs(out[1, 5] - r[1]) < 1e-5 * r[1] and max(out[1, 3], out[1, 4]) < 1e-3 * r[1]
    assert abs(out[2, 0] - r[2]) < 1e-5 * r[2] and abs(out[2, 3] - r[2]) < 1e-5 * r[2]
    with pytest.raises(T.TrackError) as e:
        T.track_band_disagreement(dev_f32(np.ones((1, 1, 1, 1, 600))),
                                  dev_f32(np.ones((1, 1, 1, 1, 600))))
    assert e.value.code == T.TRACK_EUNSUPPORTED


# ---------------------------------------------------------------- multistep scheduler (Eq. 2)
@pytest.mark.parametrize("n", [1, 3, 4096 + 3, 2_096_640])
def test_multistep_step_matches_oracle(T, n):
    rng = np.random.default_rng(n + 5)
    sig = track.schedule(4, 5.0)
    x = rng.normal(size=n).astype(np.float32)
    xd = dev_f32(x)
    state = torch.full((2 * n,), float("nan"), device=DEV)   # step 0 must not read it
    xr, st = x.astype(np.float64), None
    for i in range(4):
        v = rng.normal(size=n).astype(np.float32)
        T.track_multistep_step(xd, dev_f32(v), state, sig, i)
        T.track_sync()
        xr, st = track.multistep_update(i, xr, v, st, sig)
        assert rel_l2(xd.cpu().numpy(), xr) < 1e-6
        xr = xd.cpu().numpy().astype(np.float64)   # continue from the GPU's own values
        st = tuple(a.cpu().numpy().astype(np.float64) for a in state.view(2, n))
    with pytest.raises(T.TrackError):
        T.track_multistep_step(xd, xd, state, sig, 0)          # v aliases x
    with pytest.raises(T.TrackError):
        T.track_multistep_step(xd, dev_f32(x), state, sig, 4)  # step index out of range


# ---------------------------------------------------------------- guidance, Euler, Eq. 4
@pytest.mark.parametrize("n", [1, 3, 4096 + 3, 2_096_640])
def test_guidance_and_euler(T, n):
    rng = np.random.default_rng(n)
    fc, fu, x = (rng.normal(size=n).astype(np.float32) for _ in range(3))
    w, s0, s1 = 5.0, 0.8333333, 0.625
    p = T.track_cfg(dev_f32(fc), dev_f32(fu), w)
    T.track_sync()
    assert rel_l2(p.cpu().numpy(), track.guided(fc, fu, w)) < 1e-6
    p1 = T.track_cfg(dev_f32(fc), None, 1.0)
    assert np.array_equal(p1.cpu().numpy(), fc)                   # w = 1: exactly f_c
    xa = dev_f32(x)
    T.track_step(xa, p, s0, s1)                                   # separate
    xb = dev_f32(x)
    T.track_cfg_step(xb, dev_f32(fc), dev_f32(fu), w, s0, s1)     # fused
    T.track_sync()
    assert torch.equal(xa, xb)
    ref = track.euler_update(x, track.guided(fc, fu, w), np.float32(s0), np.float32(s1))
    assert rel_l2(xa.cpu().numpy(), ref) < 1e-6


@pytest.mark.parametrize("B,n", [(1, 1), (3, 5), (2, 4097), (8, 33_600), (1, 2_096_640)])
def test_disagreement(T, B, n):
    rng = np.random.default_rng(B * 1000 + n)
    pl = rng.normal(size=(B, n)).astype(np.float32)
    ps = (pl + 0.3 * rng.normal(size=(B, n))).astype(np.float32)
    acc = dev_f32(np.full(B, 0.25, np.float32))
    T.track_disagreement(dev_f32(pl), dev_f32(ps), acc)
    T.track_sync()
    got = acc.cpu().numpy() - 0.25                                # accumulates into the output
    ref = [track.disagreement(pl[b], ps[b]) for b in range(B)]
    assert np.max(np.abs(got - ref)) < 1e-5
    again = dev_f32(np.full(B, 0.25, np.float32))
    T.track_disagreement(dev_f32(pl), dev_f32(ps), again)
    assert torch.equal(acc, again)                                # deterministic


@pytest.mark.parametrize("B,n", [(1, 3), (3, 2_096_641), (64, 40_000), (2, 4 * 2_096_640)])
def test_disagreement_one_launch_equals_two_launches(T, B, n):
    # track_disagreement runs Eq. 4 in one launch (the last block of a sample adds
    # the partials); the allocation-free entry point runs the same partials and the
    # same fixed-order combine in two launches: the bits must agree, call after call
    # (the one-launch kernel's counters are reset by each call).
    rng = np.random.default_rng(B + n)
    pl = dev_f32(rng.normal(size=(B, n)).astype(np.float32))
    ps = dev_f32(rng.normal(size=(B, n)).astype(np.float32))
    for _ in range(3):
        one = torch.full((B,), 0.125, device=DEV)
        two = torch.full((B,), 0.125, device=DEV)
        T.track_disagreement(pl, ps, one)
        T.track_disagreement_static(pl, ps, two)
        T.track_sync()
        assert torch.equal(one, two)


@pytest.mark.parametrize("B,n", [(1, 3), (2, 4097), (1, 2_096_640), (3, 2_096_641),
                                 (4, 2_096_640)])
def test_disagreement_update_equals_separate_calls(T, B, n):
    # Calibration's per-step call: Eq. 4 and the Euler update of the trajectory by
    # p_L in one pass.  Its score must have the bits of track_disagreement and its
    # latent those of track_step, call after call; both also against the oracle.
    rng = np.random.default_rng(7 * B + n)
    pl = rng.normal(size=(B, n)).astype(np.float32)
    ps = (pl + 0.2 * rng.normal(size=(B, n))).astype(np.float32)
    x = rng.normal(size=(B, n)).astype(np.float32)
    s0, s1 = 0.8333333, 0.625
    pld, psd = dev_f32(pl), dev_f32(ps)
    xa, xb = dev_f32(x), dev_f32(x)
    acc_a = torch.full((B,), 0.5, device=DEV)
    acc_b = torch.full((B,), 0.5, device=DEV)
    for _ in range(2):
        T.track_disagreement(pld, psd, acc_a)
        T.track_step(xa, pld, s0, s1)
        T.track_disagreement_update(pld, psd, acc_b, xb, s0, s1)
        T.track_sync()
        assert torch.equal(acc_a, acc_b)
        assert torch.equal(xa, xb)
    ref_r = [track.disagreement(pl[b], ps[b]) for b in range(B)]
    assert np.max(np.abs((acc_b.cpu().numpy() - 0.5) / 2 - ref_r)) < 1e-5
    ref_x = x
    for _ in range(2):
        ref_x = track.euler_update(ref_x, pl, np.float32(s0), np.float32(s1))
    assert rel_l2(xb.cpu().numpy(), ref_x) < 1e-6
    with pytest.raises(T.TrackError):
        T.track_disagreement_update(pld, psd, acc_b, pld, s0, s1)  # x aliases p_L


def test_disagreement_special_cases(T):
    pl = np.random.default_rng(1).normal(size=(2, 1000)).astype(np.float32)
    acc = torch.zeros(2, device=DEV)
    T.track_disagreement(dev_f32(pl), dev_f32(pl), acc)
    T.track_sync()
    assert np.all(acc.cpu().numpy() == 0.0)                       # identical predictions
    acc.zero_()
    T.track_disagreement(dev_f32(pl), torch.zeros(2, 1000, device=DEV), acc)
    T.track_sync()
    assert np.allclose(acc.cpu().numpy(), 1.0, atol=1e-6)         # p_S = 0
    acc.zero_()
    T.track_disagreement(torch.zeros(2, 1000, device=DEV), dev_f32(pl), acc, eps=1e-3)
    T.track_sync()
    ref = np.linalg.norm(pl.astype(np.float64), axis=1) / 1e-3
    assert np.allclose(acc.cpu().numpy(), ref, rtol=1e-6)         # p_L = 0: eps clamp


# ---------------------------------------------------------------- on-device weights
@pytest.mark.parametrize("dtype", [0, 1])
def test_seeded_weights_equal_host_generator(T, dtype):
    wl = synth.WORKLOADS["tiny"]
    arch = wl.small
    host = T.track_model_create(arch, list(synth.make_weights(arch, 77).values()), dtype)
    seeded = T.track_model_create_seeded(arch, 77, dtype)
    x, c, u = synth.evaluation_inputs(arch, 0, 2, with_uncond=True)
    xd, cd, ud = dev_f32(x), dev_f32(c), dev_f32(u)
    a = T.track_denoise(host, xd, 600.0, cd, ud, 5.0)
    b = T.track_denoise(seeded, xd, 600.0, cd, ud, 5.0)
    T.track_sync()
    assert torch.equal(a, b)
