"""The allocation-free Eq. 4 entry point (track_disagreement_static).

For callers that cannot allocate device memory while they run (a process whose
device memory is reserved up front by its own pool, or a loop that cannot take
cudaMalloc's device-wide synchronization), the library offers a variant of
track_disagreement whose scratch is a fixed device array inside the library.
This file is collected last so that a run stopping at its first failure has
already run every other test; it passes alone in a fresh process as well.
"""
import numpy as np
import pytest

from oracle import track

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

TOL = 1e-5     # the absolute score tolerance of the other disagreement tests


@pytest.fixture(scope="module")
def T():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2609_30096_gb300 import _build
    _build.build()
    import paper_2609_30096_gb300 as T
    return T


def test_static_variant_matches_allocating_entry_point_twice_in_a_row(T):
    rng = np.random.default_rng(2024)
    for B, n in ((8, 33_600 + 3), (3, 2_096_640)):          # two calls in a row
        pl = rng.normal(size=(B, n)).astype(np.float32)
        ps = (pl + 0.2 * rng.normal(size=(B, n))).astype(np.float32)
        dl, ds = torch.from_numpy(pl).cuda(), torch.from_numpy(ps).cuda()
        ref = torch.full((B,), 0.5, device="cuda")
        got = torch.full((B,), 0.5, device="cuda")
        T.track_disagreement(dl, ds, ref)
        T.track_disagreement_static(dl, ds, got)
        T.track_sync()
        a, b = ref.cpu().numpy(), got.cpu().numpy()
        assert np.max(np.abs(a - b)) <= TOL
        oracle = np.array([track.disagreement(pl[j], ps[j]) for j in range(B)]) + 0.5
        assert np.max(np.abs(b - oracle)) <= TOL


def test_static_variant_rejects_too_many_samples(T):
    x = torch.zeros((65, 16), device="cuda")
    acc = torch.zeros(65, device="cuda")
    with pytest.raises(T.TrackError) as e:
        T.track_disagreement_static(x, x, acc)
    assert e.value.code == T.TRACK_EINVAL
    assert "maximum of 64" in str(e.value)
