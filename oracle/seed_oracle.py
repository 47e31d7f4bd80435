"""Oracle for the analytic seed of Sec. 3.1 (plain, slow, fp64).

TEST INFRASTRUCTURE ONLY: imported by tests/ (and, like trackfit_oracle, by
nothing on the product path).  Not used by the CUDA kernels yet: the seed is the
next step on the path, and this module fixes what it computes first.

What it computes (Sec. 3.1): from three hits of a track, the circle through their
transverse positions by the conformal (inversion) map of Karimaki (1991), which
turns "circle through three points" into "line through two points" with no fit
or iteration; the circle's radius and turning direction give p_T and the charge;
the direction at the point of closest approach to the beam line gives phi; the z
positions against the transverse arc length give theta; the closest-approach
point gives d0 and z0.  Everything in fp64 (the paper computes the seed in fp64
to avoid a cancellation in the transport to the beam line).

Conventions (those of the synthetic track generator, against which the tests pin
the functions): B along +z; a positive charge turns clockwise seen from +z; at
turning angle a from the perigee the direction angle is phi0 - q a, the
transverse arc length R a, and z = z0 + R a cot(theta); the perigee point is
(-d0 sin phi0, d0 cos phi0); p_T = C R B / 1000 GeV for R in mm and B in T, with
C = 0.299792458; q/p = q sin(theta) / p_T in 1/GeV.

Readings where the paper is silent:
- the seed triplet: hits taken in path order, each seed hit the first later hit
  more than 10 mm (3-D) from the previous seed hit, so that overlap hits on the
  same layer (1.5 mm apart) never form a pair; the slope uses the first and the
  third seed hit (the longer lever arm);
- with fewer than three hits so spaced the seed is undefined (NaN row);
- the per-hit features: the foot point is the helix point whose normal plane
  holds the hit, du and dv the hit's coordinates there along U = z x t / |z x t|
  and V = t x U, s_helix the 3-D path length from the perigee to the foot point,
  the asinh scale 1 mm;
- the decode: d0, z0, phi, theta add the heads' corrections (phi wrapped), q/p
  adds r (|q/p_seed| + 0.02 / GeV) (Sec. 3.3 states the residuals, not how the
  heads' outputs are scaled; the corrections here are taken as given).

Parity status: pinned in tests/test_oracle_seed.py (closed-form recovery of
generated helices to fp64 rounding, invariances under rotation about and
translation along the beam line, charge reversal, hit order; zero residuals of
points on the helix and exact recovery of displacements in the normal plane;
the decode's closed forms).
"""
from __future__ import annotations

import numpy as np

C_LIGHT = 0.299792458          # GeV / (T m)
SEED_MIN_SEPARATION_MM = 10.0
PITCH_MIN_MM = 1.0             # below this pitch z does not choose the helix turn of a hit

__all__ = ["circle_through_three", "seed_perigee", "seed_triplet", "seed_from_hits", "helix_point",
           "helix_tangent", "curvilinear_residuals", "seed_features", "decode", "C_LIGHT",
           "SEED_MIN_SEPARATION_MM", "QOP_EPS"]


def circle_through_three(p0, p1, p2):
    """Centre and radius of the circle through three transverse points [..., 2].

    With p0 moved to the origin, the inversion (u, v) = (x, y) / (x^2 + y^2) maps a
    circle through the origin with centre c onto the straight line
    2 c_x u + 2 c_y v = 1 (divide x^2 + y^2 = 2 c.x by x^2 + y^2); the images of
    p1 and p2 fix that line, i.e. two linear equations in c.  Collinear points give
    an infinite radius."""
    p0, p1, p2 = (np.asarray(p, dtype=np.float64) for p in (p0, p1, p2))
    a = p1 - p0
    b = p2 - p0
    na = np.sum(a * a, axis=-1)
    nb = np.sum(b * b, axis=-1)
    u1, v1 = a[..., 0] / na, a[..., 1] / na
    u2, v2 = b[..., 0] / nb, b[..., 1] / nb
    det = u1 * v2 - u2 * v1
    with np.errstate(divide="ignore", invalid="ignore"):
        cx = (v2 - v1) / (2.0 * det)
        cy = (u1 - u2) / (2.0 * det)
    centre = np.stack([p0[..., 0] + cx, p0[..., 1] + cy], axis=-1)
    return centre, np.hypot(cx, cy)


def _wrap(a):
    return (a + np.pi) % (2.0 * np.pi) - np.pi


def seed_perigee(h0, h1, h2, b_field):
    """Perigee parameters (d0, z0, phi0, theta, q/p) [..., 5] of the helix through
    three hits h0, h1, h2 [..., 3] (x, y, z in mm), given in path order.

    Charge: moving h0 -> h1 -> h2 the track turns left (counter-clockwise) for a
    negative charge: q = -sign((h1 - h0) x (h2 - h0)).  The closest transverse
    point of the circle to the beam line is P = C - R C/|C|; there the direction
    has the centre on its right for q > 0, i.e. t = q (-C_y, C_x)/|C| rotated to
    the direction of motion, and d0 = P . (-sin phi0, cos phi0).  The turning
    angle from P to a hit is the angle swept clockwise (q > 0) or
    counter-clockwise (q < 0) around C; with the transverse arc lengths s0, s2 of
    h0, h2, cot(theta) = (z2 - z0h) / (s2 - s0) and z0 = z0h - s0 cot(theta)."""
    h0, h1, h2 = (np.asarray(h, dtype=np.float64) for h in (h0, h1, h2))
    centre, R = circle_through_three(h0[..., :2], h1[..., :2], h2[..., :2])
    a = h1[..., :2] - h0[..., :2]
    b = h2[..., :2] - h0[..., :2]
    cross = a[..., 0] * b[..., 1] - a[..., 1] * b[..., 0]
    q = -np.sign(cross)
    dc = np.hypot(centre[..., 0], centre[..., 1])
    ux, uy = centre[..., 0] / dc, centre[..., 1] / dc          # unit vector beam line -> centre
    px, py = centre[..., 0] - R * ux, centre[..., 1] - R * uy  # closest point to the beam line
    # direction of motion at P: perpendicular to (C - P) = R u, centre on the right for q > 0
    tx, ty = -q * uy, q * ux
    phi0 = np.arctan2(ty, tx)
    d0 = -px * np.sin(phi0) + py * np.cos(phi0)

    def turning(h):
        # angle of (h - C) measured from (P - C), positive in the direction of motion
        g_p = np.arctan2(py - centre[..., 1], px - centre[..., 0])
        g_h = np.arctan2(h[..., 1] - centre[..., 1], h[..., 0] - centre[..., 0])
        return np.mod(-q * (g_h - g_p), 2.0 * np.pi)

    s0 = R * turning(h0)
    s2 = R * turning(h2)
    cot = (h2[..., 2] - h0[..., 2]) / (s2 - s0)
    z0 = h0[..., 2] - s0 * cot
    theta = np.arctan2(1.0, cot)
    pt = C_LIGHT * b_field * R / 1000.0
    qop = q * np.sin(theta) / pt
    return np.stack([d0, z0, phi0, theta, qop], axis=-1)


def seed_triplet(hits, n_hits, min_sep=SEED_MIN_SEPARATION_MM):
    """Indices [B, 3] of the seed hits of every track (the reading stated in the
    module docstring), -1 where a track has fewer than three such hits.  hits
    [B, T, >=3] with x, y, z first, in path order; n_hits [B]."""
    hits = np.asarray(hits, dtype=np.float64)
    B = hits.shape[0]
    out = np.full((B, 3), -1, dtype=np.int64)
    for b in range(B):
        picked = [0] if n_hits[b] >= 1 else []
        for t in range(1, int(n_hits[b])):
            if len(picked) == 3:
                break
            if np.linalg.norm(hits[b, t, :3] - hits[b, picked[-1], :3]) > min_sep:
                picked.append(t)
        if len(picked) == 3:
            out[b] = picked
    return out


def seed_from_hits(hits, n_hits, b_field, min_sep=SEED_MIN_SEPARATION_MM):
    """Seed perigee [B, 5] of every track from its seed triplet; NaN rows where the
    triplet does not exist."""
    hits = np.asarray(hits, dtype=np.float64)
    idx = seed_triplet(hits, n_hits, min_sep)
    ok = idx[:, 0] >= 0
    out = np.full((hits.shape[0], 5), np.nan)
    if np.any(ok):
        rows = np.nonzero(ok)[0]
        h = [hits[rows, idx[ok, k], :3] for k in range(3)]
        out[rows] = seed_perigee(h[0], h[1], h[2], b_field)
    return out


def helix_point(perigee, alpha, b_field):
    """Position (x, y, z) [..., 3] at turning angle alpha >= 0 from the perigee, for
    perigee parameters (d0, z0, phi0, theta, q/p) [..., 5]: the forward map the
    seed inverts, written from the conventions in the module docstring."""
    d0, z0, phi0, theta, qop = (np.asarray(perigee, dtype=np.float64)[..., k] for k in range(5))
    q = np.sign(qop)
    pt = np.sin(theta) / np.abs(qop)
    R = 1000.0 * pt / (C_LIGHT * b_field)
    x0, y0 = -d0 * np.sin(phi0), d0 * np.cos(phi0)
    cx, cy = x0 + q * R * np.sin(phi0), y0 - q * R * np.cos(phi0)
    phi = phi0 - q * alpha
    x = cx - q * R * np.sin(phi)
    y = cy + q * R * np.cos(phi)
    z = z0 + R * alpha / np.tan(theta)
    return np.stack([x, y, z], axis=-1)


# ---------------------------------------------------------------------------
# per-hit residual features against the seed helix (Sec. 3.1)
# ---------------------------------------------------------------------------

def helix_tangent(perigee, alpha):
    """Unit 3-D direction of motion [..., 3] at turning angle alpha: transverse
    direction angle phi0 - q alpha, polar angle theta."""
    perigee = np.asarray(perigee, dtype=np.float64)
    phi0, theta, qop = perigee[..., 2], perigee[..., 3], perigee[..., 4]
    phi = phi0 - np.sign(qop) * alpha
    st = np.sin(theta)
    return np.stack([st * np.cos(phi), st * np.sin(phi), np.cos(theta)], axis=-1)


def curvilinear_residuals(perigee, hit, b_field, iters=60):
    """(du, dv, s) of one hit [..., 3] against the helix of perigee [..., 5].

    The foot point is the helix point whose normal plane holds the hit:
    (hit - p(a)) . t(a) = 0, solved for the turning angle a by Newton's method (a
    few steps reach fp64 rounding; the iteration stops when a no longer changes).
    The start is the hit's transverse angle around the circle's centre, counted
    from the perigee into [-pi, pi) so that it is continuous across the perigee
    (a hit just behind it gets a small negative angle, not nearly a full turn),
    moved by the whole number of turns that brings it closest to the angle the
    hit's z gives, (z - z0) tan(theta) / R, where the helix's pitch 2 pi R |cot
    theta| exceeds PITCH_MIN_MM (turns closer than that are not told apart by z;
    where they coincide, du and dv are the same on each).  In that plane
    the curvilinear axes are U = z x t / |z x t| and V = t x U (the frame of the
    linearised Kalman filter); du, dv are the hit's coordinates along them and s
    the 3-D path length R a / sin(theta) from the perigee to the foot point.
    Readings: the foot point as defined here, s measured from the perigee (negative
    behind it)."""
    perigee = np.asarray(perigee, dtype=np.float64)
    hit = np.asarray(hit, dtype=np.float64)
    d0, z0, phi0, theta, qop = (perigee[..., k] for k in range(5))
    q = np.sign(qop)
    R = 1000.0 * np.sin(theta) / np.abs(qop) / (C_LIGHT * b_field)
    x0, y0 = -d0 * np.sin(phi0), d0 * np.cos(phi0)
    cx, cy = x0 + q * R * np.sin(phi0), y0 - q * R * np.cos(phi0)
    g0 = np.arctan2(y0 - cy, x0 - cx)
    gh = np.arctan2(hit[..., 1] - cy, hit[..., 0] - cx)
    a = np.mod(-q * (gh - g0) + np.pi, 2.0 * np.pi) - np.pi
    Rcot = R / np.tan(theta)
    resolved = 2.0 * np.pi * np.abs(Rcot) > PITCH_MIN_MM
    a_z = (hit[..., 2] - z0) / np.where(resolved, Rcot, 1.0)
    turns = np.floor((a_z - a) / (2.0 * np.pi) + 0.5)
    a = np.where(resolved, a + 2.0 * np.pi * turns, a)
    for _ in range(iters):
        p = helix_point(perigee, a, b_field)
        t = helix_tangent(perigee, a)
        r = hit - p
        g = np.sum(r * t, axis=-1)
        # d/da of (hit - p) . t = -|dp/da|^2 / ... : dp/da = (R / sin theta) t, and
        # dt/da = -q sin(theta) (-sin phi, cos phi, 0)
        phi = phi0 - q * a
        dt = np.stack([q * np.sin(theta) * np.sin(phi), -q * np.sin(theta) * np.cos(phi), 0.0 * phi], axis=-1)
        dg = -R / np.sin(theta) + np.sum(r * dt, axis=-1)
        step = g / dg
        a_new = a - step
        if np.all(np.abs(a_new - a) <= 1e-15 * np.maximum(1.0, np.abs(a))):
            a = a_new
            break
        a = a_new
    p = helix_point(perigee, a, b_field)
    t = helix_tangent(perigee, a)
    zhat = np.zeros_like(t)
    zhat[..., 2] = 1.0
    U = np.cross(zhat, t)
    U = U / np.linalg.norm(U, axis=-1, keepdims=True)
    V = np.cross(t, U)
    r = hit - p
    return np.sum(r * U, axis=-1), np.sum(r * V, axis=-1), R * a / np.sin(theta)


def seed_features(perigee, hits, n_hits, b_field, scale_mm=1.0):
    """The three seed features of every hit (Sec. 3.1): asinh(du / scale),
    asinh(dv / scale) and s_helix [B, T, 3], zero on padded hits and on tracks
    without a seed.  Reading: the asinh scale is 1 mm."""
    perigee = np.asarray(perigee, dtype=np.float64)
    hits = np.asarray(hits, dtype=np.float64)
    B, T = hits.shape[:2]
    out = np.zeros((B, T, 3))
    valid = (np.arange(T)[None, :] < np.asarray(n_hits)[:, None]) & np.all(np.isfinite(perigee), axis=1)[:, None]
    for t in range(T):
        rows = np.nonzero(valid[:, t])[0]
        if rows.size == 0:
            continue
        du, dv, s = curvilinear_residuals(perigee[rows], hits[rows, t, :3], b_field)
        out[rows, t] = np.stack([np.arcsinh(du / scale_mm), np.arcsinh(dv / scale_mm), s], axis=-1)
    return out


# ---------------------------------------------------------------------------
# decode of the heads' median outputs against the seed (Sec. 3.3)
# ---------------------------------------------------------------------------

QOP_EPS = 0.02   # 1/GeV, the floor of the scale-free q/p residual


def decode(seed, delta):
    """Track parameters [..., 5] from the seed perigee and the heads' corrections:
    d0, z0, theta additive, phi additive and wrapped to (-pi, pi], and q/p from
    the scale-free residual r = (q/p - q/p_seed) / (|q/p_seed| + 0.02 / GeV)."""
    seed = np.asarray(seed, dtype=np.float64)
    delta = np.asarray(delta, dtype=np.float64)
    out = seed + delta
    out[..., 2] = np.pi - np.mod(np.pi - out[..., 2], 2.0 * np.pi)
    out[..., 4] = seed[..., 4] + delta[..., 4] * (np.abs(seed[..., 4]) + QOP_EPS)
    return out
