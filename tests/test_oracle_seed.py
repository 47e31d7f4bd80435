"""Pins for the analytic-seed oracle (Sec. 3.1), no GPU: the circle through three
points against circles of known centre and radius, exact recovery of the
generator's helices from three of their points, invariances of the perigee
under rotations about and shifts along the beam line and under a mirror
reflection, the forward helix map against the generator's, and the seed triplet
reading."""
import numpy as np

from oracle import seed_oracle as S
from paper_2609_32479_gb300 import workloads as W

B_FIELD = 2.0
rng = np.random.default_rng(31)


def _helices(n, pt_range=(0.5, 100.0), seed=7, radii=(60.0, 300.0, 700.0)):
    """Generator kinematics (workloads._draw_kinematics) and exact fp64 points of
    each helix at the turning angles where it crosses the given barrel radii
    (rows of helices that reach every radius)."""
    w = W.Workload("seed", n, W.workload("large").model, pt_range=pt_range, b_field=B_FIELD)
    g = np.random.default_rng(seed)
    pt, eta, phi0, q, d0, z0 = W._draw_kinematics(g, n, w)
    theta = 2.0 * np.arctan(np.exp(-eta))
    cot = np.sinh(eta)
    R = 1000.0 * pt / (W.C_LIGHT * B_FIELD)
    x0, y0 = -d0 * np.sin(phi0), d0 * np.cos(phi0)
    cx, cy = x0 + q * R * np.sin(phi0), y0 - q * R * np.cos(phi0)
    pts, alphas = [], []
    for r in radii:
        a = W._barrel_alpha(cx, cy, R, q, phi0, r)
        x, y = W._helix_point(cx, cy, R, q, phi0, a)
        pts.append(np.stack([x, y, z0 + R * a * cot], axis=-1))
        alphas.append(a)
    truth = np.stack([d0, z0, phi0, theta, q * np.sin(theta) / pt], axis=-1)
    ok = np.all(np.isfinite(np.stack(alphas)), axis=0)
    return [p[ok] for p in pts], truth[ok], [a[ok] for a in alphas]


def _close(got, truth):
    d = got - truth
    d[:, 2] = (d[:, 2] + np.pi) % (2 * np.pi) - np.pi
    return d


def test_circle_through_three_points_of_known_circles():
    c = rng.uniform(-5e4, 5e4, (500, 2))
    R = np.exp(rng.uniform(np.log(10.0), np.log(2e5), 500))
    ang = rng.uniform(-np.pi, np.pi, (3, 500))
    p = [c + R[:, None] * np.stack([np.cos(a), np.sin(a)], axis=-1) for a in ang]
    centre, r = S.circle_through_three(*p)
    np.testing.assert_allclose(r, R, rtol=1e-8)
    assert np.all(np.abs(centre - c) <= 1e-8 * (R[:, None] + np.abs(c)))


def test_seed_recovers_generated_helices():
    """Three exact points of a helix give back the generator's perigee (d0, z0,
    phi0, theta, q/p) to fp64 rounding, at p_T from 0.5 to 100 GeV."""
    pts, truth, _ = _helices(4000)
    got = S.seed_perigee(pts[0], pts[1], pts[2], B_FIELD)
    d = _close(got, truth)
    assert np.all(np.abs(d[:, 0]) < 1e-7)             # d0, mm
    assert np.all(np.abs(d[:, 1]) < 1e-7)             # z0, mm
    assert np.all(np.abs(d[:, 2]) < 1e-10)            # phi0
    assert np.all(np.abs(d[:, 3]) < 1e-10)            # theta
    np.testing.assert_allclose(got[:, 4], truth[:, 4], rtol=1e-8)
    assert np.all(np.sign(got[:, 4]) == np.sign(truth[:, 4]))


def test_any_three_points_of_a_helix_give_the_same_seed():
    """Points of the same helices at six radii: the triplets (40, 150, 900) and
    (60, 300, 700) mm give the same perigee."""
    radii = (40.0, 60.0, 150.0, 300.0, 700.0, 900.0)
    pts, truth, _ = _helices(600, seed=9, radii=radii)
    a = S.seed_perigee(pts[1], pts[3], pts[4], B_FIELD)
    b = S.seed_perigee(pts[0], pts[2], pts[5], B_FIELD)
    d = _close(b, a)
    assert np.all(np.abs(d[:, :4]) < 1e-7)
    np.testing.assert_allclose(b[:, 4], a[:, 4], rtol=1e-8)


def test_rotation_about_the_beam_line_shifts_phi_only():
    pts, truth, _ = _helices(800, seed=11)
    beta = 0.7
    rot = np.array([[np.cos(beta), -np.sin(beta), 0.0], [np.sin(beta), np.cos(beta), 0.0], [0.0, 0.0, 1.0]])
    a = S.seed_perigee(*pts, B_FIELD)
    b = S.seed_perigee(*[p @ rot.T for p in pts], B_FIELD)
    d = _close(b, a)
    assert np.all(np.abs(d[:, [0, 1, 3]]) < 1e-7)
    assert np.all(np.abs(((b[:, 2] - a[:, 2] - beta) + np.pi) % (2 * np.pi) - np.pi) < 1e-10)
    np.testing.assert_allclose(b[:, 4], a[:, 4], rtol=1e-9)


def test_shift_along_the_beam_line_shifts_z0_only():
    pts, truth, _ = _helices(300, seed=12)
    a = S.seed_perigee(*pts, B_FIELD)
    b = S.seed_perigee(*[p + np.array([0.0, 0.0, 25.0]) for p in pts], B_FIELD)
    np.testing.assert_allclose(b[:, 1], a[:, 1] + 25.0, rtol=0, atol=1e-9)
    np.testing.assert_allclose(b[:, [0, 2, 3, 4]], a[:, [0, 2, 3, 4]], rtol=1e-9, atol=1e-12)


def test_mirror_reflection_reverses_the_charge():
    """Reflecting y -> -y reverses the turning direction: q and phi0 change sign,
    and so does d0 (the perigee point reflects with the track)."""
    pts, truth, _ = _helices(600, seed=13)
    a = S.seed_perigee(*pts, B_FIELD)
    b = S.seed_perigee(*[p * np.array([1.0, -1.0, 1.0]) for p in pts], B_FIELD)
    np.testing.assert_allclose(b[:, 4], -a[:, 4], rtol=1e-9)
    np.testing.assert_allclose(b[:, 0], -a[:, 0], rtol=0, atol=1e-8)
    assert np.all(np.abs(((b[:, 2] + a[:, 2]) + np.pi) % (2 * np.pi) - np.pi) < 1e-10)
    np.testing.assert_allclose(b[:, [1, 3]], a[:, [1, 3]], rtol=1e-9, atol=1e-9)


def test_forward_helix_map_matches_the_generator():
    pts, truth, alphas = _helices(400, seed=14)
    for p, al in zip(pts, alphas):
        np.testing.assert_allclose(S.helix_point(truth, al, B_FIELD), p, rtol=1e-12, atol=1e-9)


def test_seed_from_unsmeared_generated_tracks():
    """The generator's own fp32 hit lists, unsmeared: the seed triplet skips overlap
    hits and the seed matches the truth within the fp32 rounding of the positions."""
    w = W.workload("large", n_tracks=3000)
    w2 = W.Workload(w.name, 3000, w.model, layout=w.layout, pt_range=w.pt_range, noise_frac=0.0,
                    drop_max=0, min_hits=w.min_hits, b_field=w.b_field)
    tb = W.gen_tracks(w2, smear=False)
    got = S.seed_from_hits(tb.hits, tb.n_hits, w2.b_field)
    ok = np.all(np.isfinite(got), axis=1)
    assert ok.mean() > 0.99
    d = _close(got[ok], tb.truth[ok])
    assert np.median(np.abs(d[:, 0])) < 1e-2 and np.median(np.abs(d[:, 1])) < 1e-2
    assert np.median(np.abs(d[:, 2])) < 1e-4 and np.median(np.abs(d[:, 3])) < 1e-4
    rel = np.abs(got[ok, 4] - tb.truth[ok, 4]) / np.abs(tb.truth[ok, 4])
    assert np.median(rel) < 1e-3
    assert np.all(np.sign(got[ok, 4]) == np.sign(tb.truth[ok, 4]))


def test_seed_triplet_skips_close_hits():
    hits = np.zeros((2, 6, 5))
    hits[0, :, 0] = [30.0, 31.0, 60.0, 61.5, 90.0, 120.0]      # x; overlap pairs 1.0 and 1.5 mm apart
    hits[1, :, 0] = [30.0, 35.0, 38.0, 0.0, 0.0, 0.0]
    idx = S.seed_triplet(hits, np.array([6, 3]), min_sep=10.0)
    assert idx[0].tolist() == [0, 2, 4]
    assert idx[1].tolist() == [-1, -1, -1]
    out = S.seed_from_hits(hits, np.array([6, 3]), B_FIELD)
    assert np.all(np.isnan(out[1]))


# ---------------------------------------------------------------- per-hit features

def _frame(truth, alpha):
    """Tangent and curvilinear axes at turning angle alpha, written directly from
    the generator's helix: direction angle phi0 - q alpha, polar angle theta."""
    q = np.sign(truth[:, 4])
    phi = truth[:, 2] - q * alpha
    st, ct = np.sin(truth[:, 3]), np.cos(truth[:, 3])
    t = np.stack([st * np.cos(phi), st * np.sin(phi), ct], axis=-1)
    U = np.stack([-np.sin(phi), np.cos(phi), 0.0 * phi], axis=-1)       # z x t / |z x t|
    V = np.cross(t, U)
    return t, U, V


def test_points_on_the_helix_have_zero_residuals():
    pts, truth, alphas = _helices(500, seed=21)
    for p, al in zip(pts, alphas):
        du, dv, s = S.curvilinear_residuals(truth, p, B_FIELD)
        assert np.all(np.abs(du) < 1e-8) and np.all(np.abs(dv) < 1e-8)
        R = 1000.0 * np.sin(truth[:, 3]) / np.abs(truth[:, 4]) / (W.C_LIGHT * B_FIELD)
        np.testing.assert_allclose(s, R * al / np.sin(truth[:, 3]), rtol=1e-12)


def test_displacements_in_the_normal_plane_are_recovered():
    """A hit moved by du U + dv V off a helix point keeps that point as its foot
    point; the residuals give back (du, dv), signs included."""
    pts, truth, alphas = _helices(800, seed=22)
    for p, al in zip(pts, alphas):
        _, U, V = _frame(truth, al)
        du = rng.uniform(-5.0, 5.0, len(al))
        dv = rng.uniform(-5.0, 5.0, len(al))
        h = p + du[:, None] * U + dv[:, None] * V
        gu, gv, s = S.curvilinear_residuals(truth, h, B_FIELD)
        np.testing.assert_allclose(gu, du, rtol=0, atol=1e-9)
        np.testing.assert_allclose(gv, dv, rtol=0, atol=1e-9)


def test_looping_and_behind_the_perigee():
    """Points a turn or two along the helix (low-momentum tracks loop) and just
    behind the perigee, displaced in their normal plane: z picks the turn, so the
    foot point is the point itself and s = R a / sin(theta) with the sign and the
    whole turns; a point behind the perigee gets a small negative s, not almost a
    full turn.  Helices whose pitch 2 pi R |cot theta| is at least 100 mm (z tells
    the turns apart by more than the 5 mm displacement)."""
    g = np.random.default_rng(24)
    n = 600
    w = W.Workload("seed", n, W.workload("large").model, pt_range=(0.5, 5.0), b_field=B_FIELD)
    pt, eta, phi0, q, d0, z0 = W._draw_kinematics(g, n, w)
    theta = 2.0 * np.arctan(np.exp(-eta))
    R = 1000.0 * pt / (W.C_LIGHT * B_FIELD)
    keep = 2.0 * np.pi * R * np.abs(np.sinh(eta)) > 100.0
    pt, eta, phi0, q, d0, z0, theta, R = (v[keep] for v in (pt, eta, phi0, q, d0, z0, theta, R))
    truth = np.stack([d0, z0, phi0, theta, q * np.sin(theta) / pt], axis=-1)
    x0, y0 = -d0 * np.sin(phi0), d0 * np.cos(phi0)
    cx, cy = x0 + q * R * np.sin(phi0), y0 - q * R * np.cos(phi0)
    for base in (-0.3, 0.4, 2.0 * np.pi + 1.0, 4.0 * np.pi + 2.5):
        al = base + g.uniform(-0.2, 0.2, len(R))
        x, y = W._helix_point(cx, cy, R, q, phi0, al)
        p = np.stack([x, y, z0 + R * al * np.sinh(eta)], axis=-1)
        _, U, V = _frame(truth, al)
        du, dv = g.uniform(-5.0, 5.0, len(al)), g.uniform(-5.0, 5.0, len(al))
        gu, gv, s = S.curvilinear_residuals(truth, p + du[:, None] * U + dv[:, None] * V, B_FIELD)
        np.testing.assert_allclose(gu, du, rtol=0, atol=1e-7)
        np.testing.assert_allclose(gv, dv, rtol=0, atol=1e-7)
        np.testing.assert_allclose(s, R * al / np.sin(theta), rtol=1e-9)


def test_flat_helix_behind_the_perigee():
    """theta = pi/2 (zero pitch: every turn is the same circle, z tells none apart):
    a point just behind the perigee has the small negative s of its own turn, and
    one ahead the small positive s."""
    g = np.random.default_rng(25)
    n = 200
    R = g.uniform(500.0, 5000.0, n)
    q = np.where(g.random(n) < 0.5, -1.0, 1.0)
    phi0, d0, z0 = g.uniform(-np.pi, np.pi, n), g.normal(0.0, 0.1, n), g.normal(0.0, 50.0, n)
    theta = np.full(n, np.pi / 2)
    truth = np.stack([d0, z0, phi0, theta, q * 1000.0 / (W.C_LIGHT * B_FIELD * R)], axis=-1)
    x0, y0 = -d0 * np.sin(phi0), d0 * np.cos(phi0)
    cx, cy = x0 + q * R * np.sin(phi0), y0 - q * R * np.cos(phi0)
    for al in (g.uniform(-0.5, -0.01, n), g.uniform(0.01, 0.5, n)):
        x, y = W._helix_point(cx, cy, R, q, phi0, al)
        du, dv, s = S.curvilinear_residuals(truth, np.stack([x, y, z0], axis=-1), B_FIELD)
        assert np.all(np.abs(du) < 1e-6) and np.all(np.abs(dv) < 1e-6)
        np.testing.assert_allclose(s, R * al, rtol=1e-9)


def test_seed_features_layout_and_padding():
    pts, truth, alphas = _helices(20, seed=23)
    B = len(truth)
    hits = np.zeros((B + 1, 4, 5))
    for k in range(3):
        hits[:B, k, :3] = pts[k]
    _, U, V = _frame(truth, alphas[1])
    hits[:B, 1, :3] += 2.0 * U - 0.5 * V
    n = np.array([3] * B + [3])
    per = np.concatenate([truth, np.full((1, 5), np.nan)])
    f = S.seed_features(per, hits, n, B_FIELD)
    assert f.shape == (B + 1, 4, 3)
    np.testing.assert_allclose(f[:B, 1, 0], np.arcsinh(2.0), rtol=1e-9)
    np.testing.assert_allclose(f[:B, 1, 1], np.arcsinh(-0.5), rtol=1e-9)
    assert np.all(np.abs(f[:B, [0, 2], :2]) < 1e-8)
    assert np.all(f[:B, 3] == 0.0) and np.all(f[B] == 0.0)
    assert np.all(np.diff(f[:B, :3, 2], axis=1) > 0.0)        # path length grows along the track


# ---------------------------------------------------------------- decode

def test_decode_closed_forms():
    seed = np.array([[0.1, -3.0, 3.1, 1.2, -0.5], [0.0, 0.0, -1.0, 0.4, 0.01]])
    zero = np.zeros((2, 5))
    np.testing.assert_allclose(S.decode(seed, zero), seed, rtol=0, atol=1e-15)
    delta = np.array([[0.2, 1.0, 0.1, -0.05, 0.1], [-0.1, 0.5, 0.2, 0.01, -0.5]])
    out = S.decode(seed, delta)
    np.testing.assert_allclose(out[:, [0, 1, 3]], seed[:, [0, 1, 3]] + delta[:, [0, 1, 3]], rtol=1e-15)
    np.testing.assert_allclose(out[0, 2], 3.2 - 2.0 * np.pi, rtol=1e-14)      # wrapped into (-pi, pi]
    np.testing.assert_allclose(out[1, 2], -0.8, rtol=1e-14)
    np.testing.assert_allclose(out[0, 4], -0.5 + 0.1 * (0.5 + 0.02), rtol=1e-15)
    np.testing.assert_allclose(out[1, 4], 0.01 - 0.5 * (0.01 + 0.02), rtol=1e-14)
