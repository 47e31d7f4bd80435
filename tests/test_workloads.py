"""Synthetic input generator: helix geometry, surfaces, lengths, seeding (no GPU)."""
import numpy as np
import pytest

from paper_2609_32479_gb300 import workloads as Wl


def circumcircle(p1, p2, p3):
    """Circle through three points (textbook closed form)."""
    ax, ay = p1
    bx, by = p2
    cx, cy = p3
    d = 2 * (ax * (by - cy) + bx * (cy - ay) + cx * (ay - by))
    ux = ((ax * ax + ay * ay) * (by - cy) + (bx * bx + by * by) * (cy - ay) + (cx * cx + cy * cy) * (ay - by)) / d
    uy = ((ax * ax + ay * ay) * (cx - bx) + (bx * bx + by * by) * (ax - cx) + (cx * cx + cy * cy) * (bx - ax)) / d
    return ux, uy, np.hypot(ax - ux, ay - uy)


def test_unsmeared_hits_lie_on_helix_and_layers():
    w = Wl.workload("tiny")
    tb = Wl.gen_tracks(w, smear=False)
    radii = np.linspace(33, 1000, 10)
    h = tb.hits.astype(np.float64)
    assert np.all(tb.n_hits == 10)
    np.testing.assert_allclose(h[..., 3], np.broadcast_to(radii, h[..., 3].shape), atol=2e-3)
    np.testing.assert_allclose(np.hypot(h[..., 0], h[..., 1]), h[..., 3], rtol=1e-6)
    np.testing.assert_allclose(np.arctan2(h[..., 1], h[..., 0]), h[..., 4], atol=1e-5)
    R_expect = 1000.0 * tb.kin["pt"] / (0.299792458 * 2.0)
    for b in range(0, 256, 17):
        ux, uy, R = circumcircle(h[b, 0, :2], h[b, 4, :2], h[b, 9, :2])
        assert abs(R - R_expect[b]) / R_expect[b] < 2e-3
        # every hit on that circle
        d = np.hypot(h[b, :, 0] - ux, h[b, :, 1] - uy)
        np.testing.assert_allclose(d, R, rtol=2e-4)


def test_turning_sense_follows_charge_and_z_is_linear_in_arc_length():
    w = Wl.workload("tiny")
    tb = Wl.gen_tracks(w, smear=False)
    h = tb.hits.astype(np.float64)
    for b in range(0, 256, 5):
        cx, cy, R = tb.kin["cx"][b], tb.kin["cy"][b], tb.kin["R"][b]
        v = h[b, :, :2] - [cx, cy]
        cross = v[:-1, 0] * v[1:, 1] - v[:-1, 1] * v[1:, 0]
        # F = q v x B with B along +z turns a positive charge clockwise
        assert np.all(np.sign(cross) == -tb.kin["q"][b])
        ang = np.unwrap(np.arctan2(v[:, 1], v[:, 0]))
        s = R * np.abs(ang - ang[0])
        slope = np.polyfit(s, h[b, :, 2], 1)[0]
        assert abs(slope - np.sinh(tb.kin["eta"][b])) < 1e-4 * max(1.0, abs(slope))


def test_endcap_surfaces_and_length_range():
    w = Wl.workload("medium", n_tracks=4000)
    tb = Wl.gen_tracks(w, smear=False)
    assert tb.n_hits.min() >= 8 and tb.n_hits.max() <= 20
    assert 11.0 < tb.n_hits.mean() < 14.0
    h = tb.hits.astype(np.float64)
    T = w.model.max_hits
    valid = np.arange(T)[None, :] < tb.n_hits[:, None]
    r, z = h[..., 3][valid], h[..., 2][valid]
    on_barrel = np.min(np.abs(r[:, None] - np.linspace(33, 1000, 10)[None]), axis=1) < 2e-3
    on_disk = np.min(np.abs(np.abs(z)[:, None] - np.asarray(Wl.DISK_Z)[None]), axis=1) < 2e-3
    on_surface = on_barrel | on_disk
    # overlap hits (probability 0.5 per surface hit) sit 1.5 mm off their surface
    frac = on_surface.mean()
    assert 0.6 < frac < 0.75
    assert np.all(np.abs(z[on_barrel]) <= Wl.BARREL_HALF_LENGTH + 1e-3)
    assert np.all((r[on_disk] >= 33 - 1e-3) & (r[on_disk] <= 1000 + 1e-3))
    # pads are zero
    assert np.all(h[~valid] == 0.0)


def test_small_drops_hits_and_large_has_noise():
    tb = Wl.gen_tracks(Wl.workload("small", n_tracks=4000))
    assert set(np.unique(tb.n_hits)) == {7, 8, 9, 10}
    assert tb.hits.shape == (4000, 12, 5)
    a = Wl.gen_tracks(Wl.workload("large", n_tracks=3000), smear=False)
    b = Wl.gen_tracks(Wl.workload("medium", n_tracks=3000, ), smear=False)
    assert a.hits.shape == b.hits.shape


def test_seeding_is_reproducible():
    w = Wl.workload("small", n_tracks=512)
    a, b = Wl.gen_tracks(w), Wl.gen_tracks(w)
    np.testing.assert_array_equal(a.hits, b.hits)
    np.testing.assert_array_equal(a.n_hits, b.n_hits)
    c = Wl.gen_tracks(w, seed=17)
    assert not np.array_equal(a.hits, c.hits)
    wa, wb = Wl.gen_weights(w.model, 1), Wl.gen_weights(w.model, 1)
    np.testing.assert_array_equal(wa, wb)
    assert wa.dtype == np.float32 and wa.size == Wl.weight_count(w.model)


def test_weight_init_ranges():
    m = Wl.workload("tiny").model
    W = Wl.split_weights(m, Wl.gen_weights(m, 1))
    for name, shape, fan_in in Wl.weight_layout(m):
        if fan_in == 0:
            np.testing.assert_array_equal(W[name], 1.0)
        else:
            assert np.max(np.abs(W[name])) <= 1.0 / np.sqrt(fan_in) + 1e-7


@pytest.mark.parametrize("T", [8, 64])
def test_sweep_lengths(T):
    tb = Wl.gen_tracks(Wl.workload(f"sweep{T}", n_tracks=256), smear=False)
    assert np.all(tb.n_hits == T)
    np.testing.assert_allclose(tb.hits[0, :, 3], np.linspace(33, 1000, T), atol=2e-3)
