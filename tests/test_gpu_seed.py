"""The analytic fp64 seed, its residual features and the decode (Sec. 3.1, 3.3) on
the GPU against the seed oracle on the same seeded tracks: the seed triplet
choice bit-exactly (which tracks have a seed), the perigee and the features to
fp64 rounding of the same formulas, generated helices recovered from unsmeared
hits to the fp32 rounding of the hit coordinates, and the decode."""
import numpy as np
import pytest

from oracle import seed_oracle as S
from paper_2609_32479_gb300 import workloads as W

pytestmark = pytest.mark.gpu
torch = pytest.importorskip("torch")
B_FIELD = 2.0


@pytest.fixture(scope="module")
def T():
    import os
    from paper_2609_32479_gb300 import trackfit
    if not os.path.exists(trackfit.LIB_PATH):
        import __graft_entry__
        __graft_entry__.build()
    trackfit.load()
    return trackfit


def gpu_seed(T, hits, n_hits, features=True):
    dev = torch.device("cuda:0")
    h = torch.from_numpy(np.ascontiguousarray(hits)).to(dev)
    n = torch.from_numpy(np.ascontiguousarray(n_hits)).to(dev)
    sd = torch.full((h.shape[0], 5), -9.0, dtype=torch.float64, device=dev)
    ft = torch.full((h.shape[0], h.shape[1], 3), -9.0, dtype=torch.float32, device=dev) if features else None
    T.seed(h, n, B_FIELD, sd, ft)
    torch.cuda.synchronize()
    return sd.cpu().numpy(), (ft.cpu().numpy() if features else None)


def wrap(d):
    d = d.copy()
    d[..., 2] = (d[..., 2] + np.pi) % (2 * np.pi) - np.pi
    return d


@pytest.mark.parametrize("name,n", [("medium", 3000), ("large", 3000), ("sweep16", 2000), ("small", 2000)])
def test_seed_and_features_match_the_oracle(T, name, n):
    w = W.workload(name, n_tracks=n)
    tb = W.gen_tracks(w)
    got, feats = gpu_seed(T, tb.hits, tb.n_hits)
    ref = S.seed_from_hits(tb.hits, tb.n_hits, B_FIELD)
    # the same tracks have a seed (triplet choice is integer work: bit-exact)
    np.testing.assert_array_equal(np.isnan(got), np.isnan(ref))
    ok = ~np.isnan(ref[:, 0])
    assert ok.mean() > 0.95
    # The same fp64 formulas on both sides; the device's and numpy's fp64
    # transcendentals may differ in the last bit, which d0's cancellation
    # (d0 = -p_x sin phi0 + p_y cos phi0 with |p| up to the radius) amplifies.
    # Seeds of tracks near the beam line (|d0| < 10 mm): d0 and z0 to 1e-5 mm
    # (z0 carries the lever arm from the first hit, metres for stiff tracks;
    # 1e-5 mm is still below the fp32 rounding of a hit at 1 m), angles to
    # 1e-11 rad, q/p to 1e-9 relative.  Triplets with noise hits give
    # ill-conditioned circles: those only to 1e-6 of their scale.
    d = np.abs(wrap(got[ok] - ref[ok]))
    r = ref[ok]
    phys = np.abs(r[:, 0]) < 10.0
    tight = np.array([1e-5, 1e-5, 1e-11, 1e-11, 0.0]) + np.array([0, 0, 0, 0, 1e-9]) * np.abs(r)
    assert np.all(d[phys] <= tight[phys]), np.max(d[phys] / tight[phys], axis=0)
    loose = 1e-6 * np.maximum(np.abs(r), [1.0, 1.0, 1.0, 1.0, 1e-3])
    assert np.all(d <= loose), np.max(d / loose, axis=0)
    fref = S.seed_features(ref, tb.hits, tb.n_hits, B_FIELD)
    valid = (np.arange(w.model.max_hits)[None, :] < tb.n_hits[:, None]) & ok[:, None]
    assert np.all(feats[~valid] == 0.0)
    # asinh(du), asinh(dv) are O(1); s_helix is up to a few metres.  The foot point
    # is unique near the helix; for a hit far off it (the noise hits of the large
    # workload) the normal-plane condition has several roots and the Newton
    # iteration may settle on a different one from a last-bit difference, so
    # those hits (|du| or |dv| above 50 mm: a three-hit seed extrapolated to the
    # outer layers misses real hits by millimetres, noise hits lie hundreds of
    # millimetres off) are only required to be finite.
    fv, rv = feats[valid], fref[valid]
    near = (np.abs(np.sinh(rv[:, 0])) < 50.0) & (np.abs(np.sinh(rv[:, 1])) < 50.0)
    assert near.mean() > 0.8
    df = np.abs(fv[near] - rv[near])
    assert np.max(df[:, :2]) < 2e-6, np.max(df[:, :2])
    assert np.max(df[:, 2] / np.maximum(np.abs(rv[near][:, 2]), 1.0)) < 1e-6
    assert np.all(np.isfinite(fv))


def test_seed_recovers_unsmeared_helices(T):
    """Hits exactly on the generated helices (fp32 coordinates, no noise hits): the
    seed returns the generator's perigee within the fp32 rounding of the hits,
    with the right charge on every track."""
    w = W.workload("large", n_tracks=3000)
    w2 = W.Workload(w.name, 3000, w.model, layout=w.layout, pt_range=w.pt_range, noise_frac=0.0,
                    drop_max=0, min_hits=w.min_hits, b_field=w.b_field)
    tb = W.gen_tracks(w2, smear=False)
    got, _ = gpu_seed(T, tb.hits, tb.n_hits, features=False)
    ok = np.all(np.isfinite(got), axis=1)
    assert ok.mean() > 0.99
    d = wrap(got[ok] - tb.truth[ok])
    assert np.median(np.abs(d[:, 0])) < 1e-2 and np.median(np.abs(d[:, 1])) < 1e-2
    assert np.median(np.abs(d[:, 2])) < 1e-4 and np.median(np.abs(d[:, 3])) < 1e-4
    rel = np.abs(d[:, 4]) / np.abs(tb.truth[ok, 4])
    assert np.median(rel) < 1e-3
    assert np.all(np.sign(got[ok, 4]) == np.sign(tb.truth[ok, 4]))


def test_seed_of_short_and_invalid_tracks(T):
    w = W.workload("medium", n_tracks=64)
    tb = W.gen_tracks(w)
    n = tb.n_hits.copy()
    n[0], n[1], n[2], n[3] = 0, 1, 2, w.model.max_hits + 1
    got, feats = gpu_seed(T, tb.hits, n)
    assert np.all(np.isnan(got[:4]))
    assert np.all(feats[:4] == 0.0)
    ref = S.seed_from_hits(tb.hits[4:], n[4:], B_FIELD)
    np.testing.assert_array_equal(np.isnan(got[4:]), np.isnan(ref))


def test_decode_matches_the_oracle(T):
    rng = np.random.default_rng(4)
    B = 5000
    seed = np.stack([rng.normal(0, 0.1, B), rng.normal(0, 50, B), rng.uniform(-np.pi, np.pi, B),
                     rng.uniform(0.1, 3.0, B), rng.choice([-1, 1], B) * rng.uniform(0.01, 2.0, B)], axis=1)
    corr = rng.normal(0, 0.05, (B, 5)).astype(np.float32)
    corr[:, 2] += np.where(rng.random(B) < 0.3, 0.5, 0.0).astype(np.float32)   # some phi past +-pi
    dev = torch.device("cuda:0")
    out = torch.empty((B, 5), dtype=torch.float32, device=dev)
    T.decode(torch.from_numpy(seed).to(dev), torch.from_numpy(corr).to(dev), out)
    torch.cuda.synchronize()
    got = out.cpu().numpy().astype(np.float64)
    ref = S.decode(seed, corr.astype(np.float64))
    assert np.all(np.abs(got[:, 2]) <= np.pi + 1e-6)
    d = np.abs(wrap(got - ref))
    assert np.all(d <= 4e-7 * np.maximum(np.abs(ref), 1.0)), d.max(axis=0)


def test_seed_argument_errors(T):
    dev = torch.device("cuda:0")
    h = torch.zeros((4, 10, 5), device=dev)
    n = torch.full((4,), 5, dtype=torch.int32, device=dev)
    sd = torch.zeros((4, 5), dtype=torch.float64, device=dev)
    lib = T.load()
    s = torch.cuda.current_stream().cuda_stream
    hp, np_, sp = h.data_ptr(), n.data_ptr(), sd.data_ptr()
    assert lib.trackfit_seed(hp, 5, np_, 0, 10, 2.0, sp, None, 3, s) == T.ERR_INVALID_ARG
    assert lib.trackfit_seed(hp, 5, np_, 4, 10, 0.0, sp, None, 3, s) == T.ERR_INVALID_ARG
    assert lib.trackfit_seed(hp, 5, np_, 4, 65, 2.0, sp, None, 3, s) == T.ERR_INVALID_ARG
    assert lib.trackfit_seed(hp + 4, 5, np_, 4, 10, 2.0, sp, None, 3, s) == T.ERR_INVALID_ARG
    assert lib.trackfit_seed(hp, 2, np_, 4, 10, 2.0, sp, None, 3, s) == T.ERR_INVALID_ARG
    assert lib.trackfit_seed(hp, 5, np_, 4, 10, 2.0, sp, hp, 2, s) == T.ERR_INVALID_ARG
    assert lib.trackfit_decode(None, h.data_ptr(), 4, h.data_ptr(), s) == T.ERR_INVALID_ARG
