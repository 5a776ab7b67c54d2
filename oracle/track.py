"""The TRACK method in fp64: guidance, scheduler, disagreement, policy, calibration, sampling.

Test infrastructure only (see the package docstring).  Paper references are to
"Accelerating Video Diffusion via Training-Free Trajectory Routing" (TRACK).
"""
from __future__ import annotations

import itertools
import math

import numpy as np

# ---------------------------------------------------------------------------
# Scheduler timesteps and the scheduler update (Sec. 3.1, Eq. 2)
# ---------------------------------------------------------------------------


def schedule(n_steps: int, shift: float) -> np.ndarray:
    """Decreasing noise levels sigma_0 > ... > sigma_N as fp32 values (N+1 of them).

    Sec. 3.1 only requires a decreasing timestep sequence t_0 > ... > t_{N-1};
    the paper leaves the sampler to each pipeline.  Reading used here: the
    flow-matching grid with shift s, sigma_hat_i = 1 - i/N and
    sigma_i = s*sigma_hat_i / (1 + (s-1)*sigma_hat_i), computed in fp64 and
    exchanged as fp32 (so sigma_0 = 1 and sigma_N = 0).
    """
    if n_steps < 1:
        raise ValueError("n_steps must be >= 1")
    i = np.arange(n_steps + 1, dtype=np.float64)
    sh = 1.0 - i / n_steps
    sig = shift * sh / (1.0 + (shift - 1.0) * sh)
    return sig.astype(np.float32)


def model_timestep(sigma) -> np.float32:
    """Model timestep t_i fed to the denoiser: fp32(1000 * sigma_i) (reading; paper silent)."""
    return np.float32(np.float32(1000.0) * np.float32(sigma))


def euler_update(x, p, sigma_t, sigma_next):
    """Scheduler update S of Eq. 2 for a flow-matching velocity p, with empty history h_i.

    x_{t_{i+1}} = x_{t_i} + (sigma_{i+1} - sigma_i) * p.
    """
    x = np.asarray(x, dtype=np.float64)
    return x + (float(sigma_next) - float(sigma_t)) * np.asarray(p, dtype=np.float64)


def multistep_update(i: int, x, p, state, sigmas):
    """Scheduler update S(x_{t_i}, p, t_i, h_i) of Eq. 2 with a history h_i: a
    second-order predictor-corrector for the flow-matching ODE dx/dsigma = v.

    Sec. 3.1 lets S carry any history a multistep solver needs, and TRACK keeps
    its evolution unchanged while switching models; the pipelines' sampler
    (UniPC) is named but not written out.  Reading used here, with
    h_i = sigma_{i+1} - sigma_i and v_i = p, the guided prediction the routed
    model made at the latent x_i it was given:
      corrector (i >= 1): xc_i = xc_{i-1} + (h_{i-1} / 2) (v_{i-1} + v_i)
                          (trapezoid over [sigma_{i-1}, sigma_i]);  xc_0 = x_0;
      predictor:          x_{i+1} = xc_i + h_i v_i                       (i = 0)
                          x_{i+1} = xc_i + h_i ((1 + r/2) v_i - (r/2) v_{i-1}),
                          r = h_i / h_{i-1}                              (i >= 1)
                          (v extrapolated linearly from the last two steps).
    The one evaluation at the predicted x_i serves both the corrector of step
    i and the predictor of step i+1, so the scheme costs one denoiser call per
    step, whichever model makes it.  state = h_i = (xc_{i-1}, v_{i-1}), None
    at i = 0.  Returns (x_{i+1}, h_{i+1}) in fp64.
    """
    x = np.asarray(x, dtype=np.float64)
    v = np.asarray(p, dtype=np.float64)
    h = float(sigmas[i + 1]) - float(sigmas[i])
    if state is None:
        xc = x
        x_next = xc + h * v
    else:
        xc_prev, v_prev = state
        h_prev = float(sigmas[i]) - float(sigmas[i - 1])
        xc = xc_prev + 0.5 * h_prev * (v_prev + v)
        r = h / h_prev
        x_next = xc + h * ((1.0 + 0.5 * r) * v - 0.5 * r * v_prev)
    return x_next, (xc, v)


# ---------------------------------------------------------------------------
# Guidance (Eq. 1)
# ---------------------------------------------------------------------------


def guided(f_cond, f_uncond, w):
    """Eq. 1: p = f(x, t, empty) + w * (f(x, t, tau) - f(x, t, empty)).

    With w == 1 the unconditional branch cancels exactly; the caller may then
    pass f_uncond=None and the conditional prediction is returned unchanged.
    """
    f_cond = np.asarray(f_cond, dtype=np.float64)
    if float(w) == 1.0:
        return f_cond.copy()
    f_uncond = np.asarray(f_uncond, dtype=np.float64)
    return f_uncond + float(w) * (f_cond - f_uncond)


# ---------------------------------------------------------------------------
# Disagreement (Eq. 4) and mean score (Eq. 5)
# ---------------------------------------------------------------------------


def disagreement(p_large, p_small, eps: float = 1e-8) -> float:
    """Eq. 4: r = ||p_S - p_L||_2 / max(||p_L||_2, eps), norms over the whole latent of one sample."""
    pl = np.asarray(p_large, dtype=np.float64).ravel()
    ps = np.asarray(p_small, dtype=np.float64).ravel()
    num = math.sqrt(float(np.dot(ps - pl, ps - pl)))
    den = max(math.sqrt(float(np.dot(pl, pl))), eps)
    return num / den


def band_index(k: int, n: int) -> int:
    """|signed frequency| of DFT bin k of an n-point transform (numpy's fftfreq * n)."""
    return min(k, n - k)


def spatial_band(kh: int, kw: int, H: int, W: int) -> int:
    """Band 0/1/2 (low/mid/high) of spatial bin (kh, kw): the radius of the normalized
    frequency (|kh|/H, |kw|/W) in units of Nyquist (0.5) against 1/3 and 2/3, decided
    in integer arithmetic: rho^2 = 4 (kh^2/H^2 + kw^2/W^2)."""
    a, b = band_index(kh, H), band_index(kw, W)
    num = 4 * (a * a * W * W + b * b * H * H)   # rho^2 * H^2 W^2
    den = H * H * W * W
    if 9 * num < den:
        return 0
    if 9 * num < 4 * den:
        return 1
    return 2


def temporal_band(kf: int, F: int) -> int:
    """Band 0/1/2 of temporal bin kf: |kf|/F in units of Nyquist against 1/3 and 2/3."""
    a = band_index(kf, F)
    if 6 * a < F:
        return 0
    if 3 * a < F:
        return 1
    return 2


def band_disagreement(p_large, p_small, eps: float = 1e-8) -> np.ndarray:
    """Sec. 4.4: Eq. 4's disagreement split over frequency bands with an orthonormal
    Fourier transform, for one sample of shape [C, F, H, W].

    D = p_S - p_L is transformed over (F, H, W) per channel (orthonormal, so
    sum |D^|^2 = sum D^2); each bin's energy goes to one spatial band (radius of
    the (h, w) frequency in units of Nyquist: low < 1/3 <= mid < 2/3 <= high) and
    one temporal band (|f| frequency, same thirds).  The paper gives no band
    edges; these are the reading used.  Returns [6]: spatial low/mid/high then
    temporal low/mid/high, each sqrt(band energy) / max(||p_L||, eps), so that
    the squares of each triple add up to r^2 of Eq. 4.
    """
    pl = np.asarray(p_large, dtype=np.float64)
    d = np.asarray(p_small, dtype=np.float64) - pl
    C, F, H, W = d.shape
    e2 = np.abs(np.fft.fftn(d, axes=(1, 2, 3), norm="ortho")) ** 2
    sp = np.array([[spatial_band(kh, kw, H, W) for kw in range(W)] for kh in range(H)])
    tb = np.array([temporal_band(kf, F) for kf in range(F)])
    out = np.zeros(6)
    for band in range(3):
        out[band] = e2[:, :, sp == band].sum()
        out[3 + band] = e2[:, tb == band, :, :].sum()
    den = max(math.sqrt(float(np.dot(pl.ravel(), pl.ravel()))), eps)
    return np.sqrt(out) / den


def mean_score(r) -> np.ndarray:
    """Eq. 5: q_k = (1/M) sum_j r_{j,k}; r has shape [M, N].  Returned as fp32."""
    r = np.asarray(r, dtype=np.float64)
    M = r.shape[0]
    acc = np.zeros(r.shape[1], dtype=np.float64)
    for j in range(M):            # summed in calibration-sample order
        acc = acc + r[j]
    return (acc / M).astype(np.float32)


# ---------------------------------------------------------------------------
# Policy: relaxation (Eq. 6-7) and top-K switching (Sec. 3.2.3)
# ---------------------------------------------------------------------------


def relaxed_objective(beta, q, c0) -> float:
    """Eq. 6 objective sum_k (W_k - C0) * beta_k with W_k = q_k^2."""
    q = np.asarray(q, dtype=np.float64)
    return float(np.sum((q * q - c0) * np.asarray(beta, dtype=np.float64)))


def threshold_policy(q, c0) -> np.ndarray:
    """Eq. 7: beta_k = 1 where W_k < C0, 0 where W_k > C0 (0 chosen where W_k == C0)."""
    q = np.asarray(q, dtype=np.float64)
    return (q * q < c0).astype(np.uint8)


def topk_policy(q, k: int) -> np.ndarray:
    """Top-K switching (Sec. 3.2.3): route the K steps with the lowest q_k to the small model.

    Returns uint8[N] with 1 = small (S), 0 = large (L).  Ranking is on q itself
    (equivalent to W = q^2 for q >= 0).  Ties at the K/K+1 boundary, where the
    paper allows any optimal choice, go to the lower step index.
    """
    q = np.asarray(q, dtype=np.float32)
    n = q.shape[0]
    if not (0 <= k <= n):
        raise ValueError("K must satisfy 0 <= K <= N")
    if np.any(np.isnan(q)) or np.any(q < 0):
        raise ValueError("scores must be non-negative numbers")
    order = sorted(range(n), key=lambda i: (float(q[i]), i))
    pol = np.zeros(n, dtype=np.uint8)
    for i in order[:k]:
        pol[i] = 1
    return pol


def brute_force_topk(q, k: int) -> np.ndarray:
    """Exhaustive search over all C(N, K) subsets for the minimum of sum_{k in set} q_k^2.

    Among optimal subsets the lexicographically smallest sorted index tuple wins.
    Only for small N (test pin of ``topk_policy``).
    """
    q = [float(v) for v in np.asarray(q, dtype=np.float32)]
    n = len(q)
    best, best_set = None, None
    for combo in itertools.combinations(range(n), k):
        cost = sum(q[i] * q[i] for i in combo)
        if best is None or cost < best or (cost == best and combo < best_set):
            best, best_set = cost, combo
    pol = np.zeros(n, dtype=np.uint8)
    for i in best_set:
        pol[i] = 1
    return pol


def first_k_policy(n: int, k: int) -> np.ndarray:
    """Equal-budget baseline First-K (Sec. 4.5, Table 2): the first K steps go to the small model."""
    pol = np.zeros(n, dtype=np.uint8)
    pol[:k] = 1
    return pol


def last_k_policy(n: int, k: int) -> np.ndarray:
    """Equal-budget baseline Last-K (Sec. 4.5, Table 2): the last K steps go to the small model."""
    pol = np.zeros(n, dtype=np.uint8)
    if k:
        pol[n - k:] = 1
    return pol


def random_k_policy(n: int, k: int, seed: int) -> np.ndarray:
    """Equal-budget baseline Random-K (Sec. 4.5, Table 2): a uniformly random K-subset.

    The random numbers are an input of the method: partial Fisher-Yates shuffle of
    0..n-1 whose i-th swap partner is i + (u_i mod (n - i)), u_i being output i of
    a SplitMix64 stream (Steele, Lea and Flood 2014) started at mix64(seed).
    """
    if not (0 <= k <= n):
        raise ValueError("K must satisfy 0 <= K <= N")
    mask = (1 << 64) - 1

    def mix64(z):
        z &= mask
        z = ((z ^ (z >> 30)) * 0xBF58476D1CE4E5B9) & mask
        z = ((z ^ (z >> 27)) * 0x94D049BB133111EB) & mask
        return z ^ (z >> 31)

    state = mix64(seed)
    perm = list(range(n))
    for i in range(k):
        u = mix64(state + (i + 1) * 0x9E3779B97F4A7C15)
        j = i + u % (n - i)
        perm[i], perm[j] = perm[j], perm[i]
    pol = np.zeros(n, dtype=np.uint8)
    pol[perm[:k]] = 1
    return pol


# ---------------------------------------------------------------------------
# Denoiser evaluation, calibration (Sec. 3.2.1) and routed sampling (Eq. 3)
# ---------------------------------------------------------------------------


def guided_prediction(model, x, sigma, cond, uncond, w, counter=None):
    """p_m(x_t, t) of Eq. 1 for one sample, evaluating f_m on tau (and on the negative prompt if w != 1)."""
    t = model_timestep(sigma)
    f_c = model.forward(x, t, cond)
    if counter is not None:
        counter[model.name] = counter.get(model.name, 0) + 1
    if float(w) == 1.0:
        return guided(f_c, None, w)
    f_u = model.forward(x, t, uncond)
    if counter is not None:
        counter[model.name] += 1
    return guided(f_c, f_u, w)


def calibrate(large, small, x_T, conds, unconds, w, sigmas, eps: float = 1e-8):
    """Reference-trajectory calibration (Sec. 3.2.1) followed by Eq. 4 scoring.

    For every calibration sample j the trajectory is rolled out with the large
    model only.  Before each update both models are evaluated on the same
    latent x_{t_k}, timestep, conditioning and guidance; r[j, k] records their
    relative disagreement and the large model's prediction advances x.
    Returns (r [M, N] float64, final latents [M, ...] float64).
    """
    M = len(x_T)
    N = len(sigmas) - 1
    r = np.zeros((M, N), dtype=np.float64)
    finals = []
    for j in range(M):
        x = np.asarray(x_T[j], dtype=np.float64)
        u = None if unconds is None else unconds[j]
        for k in range(N):
            p_l = guided_prediction(large, x, sigmas[k], conds[j], u, w)
            p_s = guided_prediction(small, x, sigmas[k], conds[j], u, w)
            r[j, k] = disagreement(p_l, p_s, eps)
            x = euler_update(x, p_l, sigmas[k], sigmas[k + 1])
        finals.append(x)
    return r, np.stack(finals)


def sample_routed_multistep(large, small, policy, x_T, cond, uncond, w, sigmas, counter=None):
    """Eq. 3 with the multistep scheduler: the history h_i evolves exactly as in
    an all-large run, whichever model supplied each p (Sec. 3.1)."""
    x = np.asarray(x_T, dtype=np.float64)
    state = None
    for i in range(len(sigmas) - 1):
        m = small if policy[i] else large
        p = guided_prediction(m, x, sigmas[i], cond, uncond, w, counter)
        x, state = multistep_update(i, x, p, state, sigmas)
    return x


def sample_routed(large, small, policy, x_T, cond, uncond, w, sigmas, counter=None):
    """Eq. 3: x_{t_{i+1}} = S(x_{t_i}, p_{pi(i)}(x_{t_i}, t_i), t_i, h_i), one denoiser per step."""
    x = np.asarray(x_T, dtype=np.float64)
    for i in range(len(sigmas) - 1):
        m = small if policy[i] else large
        p = guided_prediction(m, x, sigmas[i], cond, uncond, w, counter)
        x = euler_update(x, p, sigmas[i], sigmas[i + 1])
    return x
