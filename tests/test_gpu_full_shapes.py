"""Kernel parity at the full sizes of the 14B/1.3B configurations, on sampled outputs.

The 480p pair (32760 tokens, CFG: two sequences per forward), the 720p pair
(75600 tokens, one sequence) and the serving batch (eight sequences of 32760
tokens, 262080 GEMM rows: output offsets past 2^31 elements) use the 14B
shapes d 5120, 40 heads of 128, FFN 13824, and the 1.3B shapes d 1536, FFN
8960.  The inputs are seeded normal draws made on the device by torch's
generator (plumbing, not this library); the oracle recomputes sampled rows
in fp64 from host copies of exactly the values the kernels read.  Serving
inputs repeat a 32760-row block, so the oracle for any row is the oracle of
its row in the block.
"""
import numpy as np
import pytest

from oracle import dit

torch = pytest.importorskip("torch")
pytestmark = [pytest.mark.gpu, pytest.mark.slow]


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
    return float(np.linalg.norm(a - b) / max(np.linalg.norm(b), 1e-300))


def randn_bf16(gen, *shape, scale=1.0):
    return (torch.randn(*shape, device="cuda", generator=gen) * scale).to(torch.bfloat16)


def host(t):
    return t.float().cpu().numpy()


def sample_rows(rng, M, n=40):
    edge = [0, 1, 127, 128, M - 129, M - 128, M - 2, M - 1]
    return np.unique(np.concatenate([edge, rng.choice(M, n, replace=False)]))


N480, N720 = 32760, 75600
D14, F14, D13, F13 = 5120, 13824, 1536, 8960

# (label, base rows, repeats, N, K, epilogue name)
GEMM_FULL = [
    ("480p 14B qkv", N480, 1, 3 * D14, D14, "store"),
    ("480p 14B ffn_up", N480, 1, F14, D14, "gelu"),
    ("480p 14B ffn_down", N480, 1, D14, F14, "resid_gate"),
    ("480p 1.3B ffn_down", N480, 1, D13, F13, "resid_gate"),
    ("720p 14B qkv", N720, 1, 3 * D14, D14, "store"),
    ("serving 14B qkv", N480, 8, 3 * D14, D14, "store"),
    ("serving 14B out_proj", N480, 8, D14, D14, "resid_gate"),
]


@pytest.mark.parametrize("label,base,reps,N,K,epi", GEMM_FULL, ids=[g[0] for g in GEMM_FULL])
def test_linear_bf16_full_size(T, label, base, reps, N, K, epi):
    gen = torch.Generator(device="cuda").manual_seed(base + N + K)
    rng = np.random.default_rng(N * 3 + K)
    Xb = randn_bf16(gen, base, K)
    X = Xb.repeat(reps, 1) if reps > 1 else Xb
    M = base * reps
    W = randn_bf16(gen, N, K, scale=K ** -0.5)
    b = torch.randn(N, device="cuda", generator=gen) * 0.1
    gate = torch.randn(N, device="cuda", generator=gen)
    code = {"store": T.EPI_STORE, "gelu": T.EPI_GELU, "resid_gate": T.EPI_RESID_GATE}[epi]
    if epi == "resid_gate":
        out = torch.zeros(M, N, device="cuda")
        T.track_linear(T.BF16, X, W, b, code, out, gate=gate)
    else:
        out = torch.zeros(M, N, device="cuda", dtype=torch.bfloat16)
        T.track_linear(T.BF16, X, W, b, code, out)
    T.track_sync()
    rows = sample_rows(rng, M)
    got = host(out[torch.from_numpy(rows).cuda()])
    del out
    ref = dit.linear(host(Xb[torch.from_numpy(rows % base).cuda()]), host(W), host(b))
    if epi == "gelu":
        ref = dit.gelu_tanh(ref)
    if epi == "resid_gate":
        ref = ref * host(gate)
        assert rel_l2(got, ref) < 2e-5, label
    else:
        assert rel_l2(got, ref) < 4e-3, label
        scale = np.sqrt(np.mean(ref ** 2))
        assert np.all(np.abs(got - ref) <= 8e-3 * np.abs(ref) + 2e-3 * scale), label


# (label, S in the block, repeats, H, Lq, Lk)
ATTN_FULL = [
    ("480p 14B self, CFG pair", 2, 1, 40, N480, N480),
    ("480p 14B cross, CFG pair", 2, 1, 40, N480, 512),
    ("720p 14B self", 1, 1, 40, N720, N720),
    ("serving 14B self", 2, 4, 40, N480, N480),
]


@pytest.mark.parametrize("label,S0,reps,H,Lq,Lk", ATTN_FULL, ids=[a[0] for a in ATTN_FULL])
def test_attention_bf16_full_size(T, label, S0, reps, H, Lq, Lk):
    hd = 128
    gen = torch.Generator(device="cuda").manual_seed(Lq + Lk + S0 * reps)
    rng = np.random.default_rng(Lq + Lk)
    Qb, Kb, Vb = (randn_bf16(gen, S0, H, L, hd) for L in (Lq, Lk, Lk))
    Q, K, V = ((t.repeat(reps, 1, 1, 1) if reps > 1 else t) for t in (Qb, Kb, Vb))
    S = S0 * reps
    O = torch.zeros(S, Lq, H, hd, device="cuda", dtype=torch.bfloat16)
    T.track_attention(T.BF16, Q, K, V, O)
    T.track_sync()
    for s, h in ((0, 0), (S - 1, H - 1), (S // 2, 17)):
        rows = sample_rows(rng, Lq, 24)
        ridx = torch.from_numpy(rows).cuda()
        got = host(O[s, ridx, h])
        sb = s % S0
        ref = dit.attention(host(Qb[sb, h, ridx]), host(Kb[sb, h]), host(Vb[sb, h]))
        assert rel_l2(got, ref) < 1e-2, (label, s, h)


# ---------------------------------------------------------------- one 14B block, full 480p
@pytest.fixture(scope="module")
def block14(T):
    """The 14B architecture cut to one block (every kernel shape of the full model
    occurs in each block) at the 480p latent: the library's model from on-device
    seeded weights, and the oracle's from the host generator."""
    import dataclasses

    import synth
    arch = dataclasses.replace(synth.WORKLOADS["wan480"].large, layers=1)
    seed = synth.SEED_LARGE
    m = T.track_model_create_seeded(arch, seed, T.BF16)
    o = dit.DiT(arch, synth.make_weights(arch, seed), "bf16")
    yield arch, m, o
    m.close()


@pytest.mark.parametrize("batch", [1, 4], ids=["480p CFG pair", "serving: 4 seeds, 8 sequences"])
def test_14b_block_guided_prediction_full_480p(T, block14, batch):
    """Guided prediction (Eq. 1, CFG 5) of one 14B-shape block over all 32760 tokens,
    checked at sampled tokens of the last seed against the oracle's forward at those
    tokens (its self-attention reads every token's keys and values)."""
    import synth
    from oracle import track
    arch, m, o = block14
    x, c, u = synth.evaluation_inputs(arch, 0, batch, with_uncond=True)
    sig = track.schedule(50, 5.0)
    t = float(track.model_timestep(sig[10]))
    v = T.track_denoise(m, torch.from_numpy(x).cuda(), t, torch.from_numpy(c).cuda(),
                        torch.from_numpy(u).cuda(), 5.0)
    T.track_sync()
    j = batch - 1
    got_tok = dit.patchify(v[j].cpu().numpy().astype(np.float64), arch.patch)
    rng = np.random.default_rng(batch)
    rows = sample_rows(rng, arch.tokens, 24)
    fc = o.forward_at_tokens(x[j], np.float32(t), c[j], rows)
    fu = o.forward_at_tokens(x[j], np.float32(t), u[j], rows)
    ref = track.guided(fc, fu, 5.0)
    assert rel_l2(got_tok[rows], ref) < 2e-2
