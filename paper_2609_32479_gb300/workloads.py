"""Named workloads and seeded synthetic inputs for the track-fit encoder.

This module is the one place that both the CUDA path (through the C-ABI) and the
CPU oracle take their inputs from.  It holds configuration numbers, the
synthetic helix-hit generator and the random-init weight generator; it holds
none of the encoder's arithmetic (no normalisation, Fourier map, projection,
scan, pooling or head).

Stand-in for the paper's data: the paper trains and evaluates on ColliderML
single-muon samples on the Open Data Detector (Sec. 2): hits ordered by
measurement time, 6-20 hits per track, 13 on average (Sec. 3.5).  Those samples
and the trained weights are not available, so every workload here is seeded
synthetic helix tracks in a uniform solenoid field, with random-init weights.

Readings of the paper's detector and sample description:
  * field B_z = 2 T; helix radius R[mm] = 1000 * pT[GeV] / (0.299792458 * B[T]);
  * 10 barrel layers at radii linspace(33, 1000); tiny/small/sweep barrels are
    unbounded cylinders, medium/large barrels have half-length 600 mm plus 7
    disks per side at |z| = 600, 1000, ..., 3000 mm (annulus r in [33, 1000]);
  * one hit per crossed surface, plus with p = 0.5 an overlap hit 1.5 mm
    further along the track (medium/large), so lengths reach 20 and the mean
    is about 12.5 (the paper's tracks have 13 hits on average, Sec. 3.5);
  * tracks with fewer than 8 hits are redrawn, longer ones truncated to 20;
  * Gaussian smearing 10 um on r*phi and z (barrel), on x and y (disks);
    r and phi are recomputed from the smeared x, y in fp64, stored fp32;
  * hits ordered by path length along the helix (the time order of Sec. 2);
  * small drops k ~ U{0..3} hits at uniformly chosen positions;
  * large replaces each hit with p = 0.05 by a uniform point on the same surface;
  * sweep: T barrel layers at radii linspace(33, 1000, T), no padding.
"""
from __future__ import annotations

import dataclasses
import math
from typing import Dict, List, Optional, Tuple

import numpy as np

# ---------------------------------------------------------------------------
# configuration
# ---------------------------------------------------------------------------

PRECISION_FP32 = 0
PRECISION_BF16 = 1
PRECISION_FP16 = 2
POOL_MEAN = 0
POOL_ENDPOINTS = 1
TOPOLOGY_MERGE = 0      # gated merge + MLP into a d_model residual stream
TOPOLOGY_CONCAT = 1     # Sec. 3.2: concatenated states into the next layer
TOPOLOGY_ATTENTION = 2  # App. A.3: Transformer encoder layers (pre-norm attention + MLP)

N_FEATURES = 5          # (x, y, z, r, phi) per hit
N_FOURIER = 16          # Sec. 3.2: "16 scales"
HEAD_HIDDEN = 128       # Sec. 3.2: head hidden width 128
N_QUANTILES = 7         # Sec. 3.2/3.3: 7 quantiles per parameter
N_PARAMS = 5            # (d0, z0, phi, theta, q/p)

# fixed min-max constants (x, y, z [mm], r [mm], phi [rad]); fixed numbers, not
# batch statistics, so a track's output does not depend on its batch.
FEAT_MIN = (-1100.0, -1100.0, -3100.0, 0.0, -math.pi)
FEAT_MAX = (1100.0, 1100.0, 3100.0, 1100.0, math.pi)
# Fourier scales s_k = 2^(k/3), k = 0..15; the feature argument is pi * s_k * u
FOURIER_SCALE = tuple(float(np.float32(2.0 ** (k / 3.0))) for k in range(N_FOURIER))


@dataclasses.dataclass(frozen=True)
class ModelConfig:
    """Encoder shape; mirrors trackfit_config_t in include/trackfit.h."""
    max_hits: int
    d_model: int
    d_hidden: int
    n_layers: int
    precision: int = PRECISION_FP32
    pool: int = POOL_MEAN
    topology: int = TOPOLOGY_MERGE
    n_heads: int = 4
    head_hidden: int = HEAD_HIDDEN
    n_quantiles: int = N_QUANTILES
    n_features: int = N_FEATURES
    n_fourier: int = N_FOURIER
    feat_min: Tuple[float, ...] = FEAT_MIN
    feat_max: Tuple[float, ...] = FEAT_MAX
    fourier_scale: Tuple[float, ...] = FOURIER_SCALE
    rms_eps: float = 1e-6

    @property
    def embed_dim(self) -> int:
        return 2 * self.n_features * self.n_fourier

    @property
    def proj_dim(self) -> int:
        """Rows of the per-layer input projection: z_f, n_f, z_b, n_b (and, MERGE, the
        gate); q, k, v for the Transformer."""
        if self.topology == TOPOLOGY_ATTENTION:
            return 3 * self.d_model
        return 4 * self.d_hidden + (self.d_model if self.topology == TOPOLOGY_MERGE else 0)

    @property
    def pooled_dim(self) -> int:
        if self.pool == POOL_MEAN and self.topology in (TOPOLOGY_MERGE, TOPOLOGY_ATTENTION):
            return self.d_model
        return 2 * self.d_hidden

    @property
    def n_out(self) -> int:
        return N_PARAMS * self.n_quantiles

    def with_(self, **kw) -> "ModelConfig":
        return dataclasses.replace(self, **kw)


@dataclasses.dataclass(frozen=True)
class Workload:
    """A named workload: batch, track generator settings and encoder shape."""
    name: str
    n_tracks: int
    model: ModelConfig
    layout: str = "barrel"          # "barrel" | "barrel_endcap" | "sweep"
    pt_range: Tuple[float, float] = (1.0, 10.0)
    noise_frac: float = 0.0
    drop_max: int = 0
    min_hits: int = 8
    n_barrel: int = 10
    track_seed: int = 0
    weight_seed: int = 1
    b_field: float = 2.0


def _model(T, D, L, prec):
    return ModelConfig(max_hits=T, d_model=D, d_hidden=(3 * D) // 2, n_layers=L, precision=prec)


WORKLOADS: Dict[str, Workload] = {
    "tiny": Workload("tiny", 256, _model(10, 32, 2, PRECISION_FP32), min_hits=10),
    "small": Workload("small", 16384, _model(12, 64, 4, PRECISION_FP32), drop_max=3, min_hits=10),
    "medium": Workload("medium", 262144, _model(24, 128, 6, PRECISION_BF16), layout="barrel_endcap"),
    "large": Workload("large", 1048576, _model(24, 256, 8, PRECISION_BF16), layout="barrel_endcap",
                      pt_range=(0.5, 100.0), noise_frac=0.05),
}
for _T in (8, 16, 32, 64):
    WORKLOADS[f"sweep{_T}"] = Workload(f"sweep{_T}", 1048576, _model(_T, 128, 6, PRECISION_BF16),
                                       layout="sweep", n_barrel=_T, min_hits=_T)
SWEEP_BATCHES = (4096, 16384, 65536, 262144, 1048576)

# The paper's model (Sec. 3.2): 15 features per hit, d_model 128, two layers of
# hidden width 192, the concatenation topology, endpoint readout; fp16 operands
# (Sec. 3.5).  Its 12 measured features are "position, derived angles, and
# detector identifiers" (Sec. 2); the list is not given, so here: x, y, z, r, phi,
# the polar angle theta = atan2(r, z), eta = asinh(z / r), the distance
# rho = |(r, z)|, cos phi, sin phi, the surface kind (barrel 0, disk 1) and the
# surface's index within its kind; the last three are the seed's residual
# features (asinh du, asinh dv, s_helix, Sec. 3.1), computed by the seed.
PAPER_FEATURES = ("x", "y", "z", "r", "phi", "theta", "eta", "rho", "cos_phi", "sin_phi", "surface_kind",
                  "surface_index", "asinh_du", "asinh_dv", "s_helix")
PAPER_FEAT_MIN = (-1100.0, -1100.0, -3100.0, 0.0, -math.pi, 0.0, -5.0, 0.0, -1.0, -1.0, 0.0, 0.0, -8.0, -8.0, 0.0)
PAPER_FEAT_MAX = (1100.0, 1100.0, 3100.0, 1100.0, math.pi, math.pi, 5.0, 3300.0, 1.0, 1.0, 1.0, 9.0, 8.0, 8.0,
                  4000.0)
WORKLOADS["paper"] = Workload(
    "paper", 131072,
    ModelConfig(max_hits=24, d_model=128, d_hidden=192, n_layers=2, precision=PRECISION_FP16, pool=POOL_ENDPOINTS,
                topology=TOPOLOGY_CONCAT, n_features=15, feat_min=PAPER_FEAT_MIN, feat_max=PAPER_FEAT_MAX),
    layout="barrel_endcap", pt_range=(1.0, 100.0))
# The Transformer of the encoder comparison (App. A.3, Tab. A.1): the paper's
# features, embedding and quantile head around three pre-norm layers of 4-head
# attention over each track's hits and an MLP of hidden width 288, mean pooled;
# 520,579 weights, within 3 % of the paper-shaped minGRU model's 527,011 (the
# paper matches its encoders' parameter counts to 3 %).
WORKLOADS["transformer"] = dataclasses.replace(
    WORKLOADS["paper"], name="transformer",
    model=WORKLOADS["paper"].model.with_(d_hidden=288, n_layers=3, pool=POOL_MEAN, topology=TOPOLOGY_ATTENTION,
                                         n_heads=4))


def workload(name: str, n_tracks: Optional[int] = None, **model_kw) -> Workload:
    w = WORKLOADS[name]
    if n_tracks is not None:
        w = dataclasses.replace(w, n_tracks=int(n_tracks))
    if model_kw:
        w = dataclasses.replace(w, model=w.model.with_(**model_kw))
    return w


# ---------------------------------------------------------------------------
# weight blob (fp32, PyTorch [out][in] order)
# ---------------------------------------------------------------------------

def weight_layout(cfg: ModelConfig) -> List[Tuple[str, Tuple[int, ...], int]]:
    """(name, shape, fan_in) of every tensor, in blob order.  fan_in = 0 marks a
    norm gain (initialised to 1)."""
    D, H, E, P = cfg.d_model, cfg.d_hidden, cfg.embed_dim, cfg.pooled_dim
    Hh, Q = cfg.head_hidden, cfg.n_out
    out = [("emb.w1", (D, E), E), ("emb.b1", (D,), E), ("emb.w2", (D, D), D), ("emb.b2", (D,), D)]
    for l in range(cfg.n_layers):
        p = f"layer{l}."
        if cfg.topology == TOPOLOGY_CONCAT:
            I = D if l == 0 else 2 * H
            out += [(p + "w_in", (4 * H, I), I), (p + "b_in", (4 * H,), I)]
            continue
        if cfg.topology == TOPOLOGY_ATTENTION:
            out += [(p + "g1", (D,), 0), (p + "w_qkv", (3 * D, D), D), (p + "b_qkv", (3 * D,), D),
                    (p + "w_o", (D, D), D), (p + "b_o", (D,), D), (p + "g2", (D,), 0),
                    (p + "w1", (H, D), D), (p + "b1", (H,), D), (p + "w2", (D, H), H), (p + "b2", (D,), H)]
            continue
        out += [(p + "g", (D,), 0), (p + "w_in", (4 * H + D, D), D), (p + "b_in", (4 * H + D,), D),
                (p + "w_m", (D, 2 * H), 2 * H), (p + "b_m", (D,), 2 * H),
                (p + "w1", (D, D), D), (p + "b1", (D,), D), (p + "w2", (D, D), D), (p + "b2", (D,), D)]
    out += [("head.g", (P,), 0), ("head.w1", (Hh, P), P), ("head.b1", (Hh,), P),
            ("head.w2", (Q, Hh), Hh), ("head.b2", (Q,), Hh)]
    return out


def weight_count(cfg: ModelConfig) -> int:
    return sum(int(np.prod(s)) for _, s, _ in weight_layout(cfg))


def gen_weights(cfg: ModelConfig, seed: int = 1) -> np.ndarray:
    """Random-init weights: U(+-1/sqrt(fan_in)) for matrices and biases, gains 1,
    drawn in blob order from PCG64(seed).  Returns a flat fp32 blob."""
    rng = np.random.Generator(np.random.PCG64(seed))
    parts = []
    for _, shape, fan_in in weight_layout(cfg):
        n = int(np.prod(shape))
        if fan_in == 0:
            parts.append(np.ones(n, dtype=np.float64))
        else:
            k = 1.0 / math.sqrt(fan_in)
            parts.append(rng.uniform(-k, k, size=n))
    return np.concatenate(parts).astype(np.float32)


def split_weights(cfg: ModelConfig, blob: np.ndarray) -> Dict[str, np.ndarray]:
    """View the flat blob as named tensors (no arithmetic, only slicing)."""
    out, off = {}, 0
    for name, shape, _ in weight_layout(cfg):
        n = int(np.prod(shape))
        out[name] = blob[off:off + n].reshape(shape)
        off += n
    if off != blob.size:
        raise ValueError(f"weight blob has {blob.size} values, layout needs {off}")
    return out


def join_weights(cfg: ModelConfig, tensors: Dict[str, np.ndarray]) -> np.ndarray:
    return np.concatenate([np.asarray(tensors[n], dtype=np.float32).reshape(-1)
                           for n, _, _ in weight_layout(cfg)])


# ---------------------------------------------------------------------------
# helix hit generator
# ---------------------------------------------------------------------------

BARREL_R_MIN, BARREL_R_MAX = 33.0, 1000.0
BARREL_HALF_LENGTH = 600.0
DISK_Z = tuple(600.0 + 400.0 * i for i in range(7))
SMEAR_MM = 0.010
OVERLAP_P = 0.5
OVERLAP_MM = 1.5
MAX_TRACK_HITS = 20
C_LIGHT = 0.299792458


@dataclasses.dataclass
class TrackBatch:
    hits: np.ndarray      # [B, T, 5] float32, pads zero
    n_hits: np.ndarray    # [B] int32
    kind: np.ndarray      # [B, T] int8: the hit's surface, 0 barrel, 1 disk, -1 padding
    truth: np.ndarray     # [B, 5] float64: d0, z0, phi, theta, q/p
    kin: Dict[str, np.ndarray]   # per-track pT, eta, q, R and helix centre (generator tests)


def _wrap(a):
    return np.mod(a + np.pi, 2.0 * np.pi) - np.pi


def _helix_point(cx, cy, R, q, phi0, alpha):
    """Transverse point after turning angle alpha (>=0) along the helix.

    A positive charge in +B_z turns clockwise seen from +z, so the direction
    angle is phi0 - q*alpha and the centre lies on the right of the start
    direction for q > 0."""
    phi = phi0 - q * alpha
    return cx - q * R * np.sin(phi), cy + q * R * np.cos(phi)


def _barrel_alpha(cx, cy, R, q, phi0, r_layer):
    """Smallest turning angle at which the transverse circle crosses radius r_layer
    (NaN where it never does)."""
    dc = np.hypot(cx, cy)
    w = (r_layer ** 2 - dc ** 2 - R ** 2) / (2.0 * R * dc)
    ok = np.abs(w) <= 1.0
    acw = np.arccos(np.clip(w, -1.0, 1.0))
    beta = np.arctan2(cy, cx)
    # angle of (start - centre): start = centre - q*R*(sin phi0, -cos phi0)
    gamma0 = np.arctan2(q * np.cos(phi0), -q * np.sin(phi0))
    d0 = gamma0 - beta
    # the centre-to-point angle moves as gamma0 - q*alpha
    a1 = np.mod(q * (d0 - acw), 2.0 * np.pi)
    a2 = np.mod(q * (d0 + acw), 2.0 * np.pi)
    return np.where(ok, np.minimum(a1, a2), np.nan)


def _draw_kinematics(rng, n, w: Workload):
    lo, hi = w.pt_range
    pt = np.exp(rng.uniform(np.log(lo), np.log(hi), n))
    eta = rng.uniform(-2.5, 2.5, n)
    phi0 = rng.uniform(-np.pi, np.pi, n)
    q = np.where(rng.random(n) < 0.5, -1.0, 1.0)
    d0 = rng.normal(0.0, 0.1, n)
    z0 = rng.normal(0.0, 50.0, n)
    return pt, eta, phi0, q, d0, z0


def _gen_raw(rng, n, w: Workload):
    """Draw n tracks; return per-track kinematics and a ragged hit list (padded
    arrays [n, S] with NaN where a surface is not hit), sorted by path length."""
    pt, eta, phi0, q, d0, z0 = _draw_kinematics(rng, n, w)
    theta = 2.0 * np.arctan(np.exp(-eta))
    cot = np.sinh(eta)
    R = 1000.0 * pt / (C_LIGHT * w.b_field)
    x0, y0 = -d0 * np.sin(phi0), d0 * np.cos(phi0)
    cx, cy = x0 + q * R * np.sin(phi0), y0 - q * R * np.cos(phi0)

    if w.layout == "sweep":
        radii = np.linspace(BARREL_R_MIN, BARREL_R_MAX, w.n_barrel)
    else:
        radii = np.linspace(BARREL_R_MIN, BARREL_R_MAX, 10)
    bounded = w.layout == "barrel_endcap"

    # transverse turning angle at which the track leaves r = BARREL_R_MAX
    a_out = _barrel_alpha(cx, cy, R, q, phi0, BARREL_R_MAX)
    a_out = np.where(np.isnan(a_out), np.inf, a_out)

    alphas, kinds = [], []      # kind 0 = barrel, 1 = disk
    for r in radii:
        a = _barrel_alpha(cx, cy, R, q, phi0, r)
        z = z0 + R * a * cot
        if bounded:
            a = np.where(np.abs(z) <= BARREL_HALF_LENGTH, a, np.nan)
        alphas.append(a)
        kinds.append(0)
    if bounded:
        for zd in DISK_Z:
            zt = np.where(cot >= 0.0, zd, -zd)
            with np.errstate(divide="ignore", invalid="ignore"):
                a = (zt - z0) / (cot * R)
            a = np.where((a > 0.0) & (a <= a_out), a, np.nan)
            px, py = _helix_point(cx, cy, R, q, phi0, np.nan_to_num(a))
            rr = np.hypot(px, py)
            a = np.where((rr >= BARREL_R_MIN) & (rr <= BARREL_R_MAX), a, np.nan)
            alphas.append(a)
            kinds.append(1)
    A = np.stack(alphas, axis=1)                          # [n, S]
    K = np.broadcast_to(np.asarray(kinds, dtype=np.int8), A.shape).copy()
    if bounded:
        # overlap hits: 1.5 mm further along the 3-D path
        extra = rng.random(A.shape) < OVERLAP_P
        dA = OVERLAP_MM * np.sin(theta)[:, None] / R[:, None]
        A2 = np.where(extra & ~np.isnan(A), A + dA, np.nan)
        A = np.concatenate([A, A2], axis=1)
        K = np.concatenate([K, K], axis=1)
    order = np.argsort(np.where(np.isnan(A), np.inf, A), axis=1, kind="stable")
    A = np.take_along_axis(A, order, axis=1)
    K = np.take_along_axis(K, order, axis=1)
    kin = dict(pt=pt, eta=eta, phi0=phi0, q=q, d0=d0, z0=z0, theta=theta, cot=cot, R=R, cx=cx, cy=cy)
    return kin, A, K


def _positions(kin, A, K, rng, w: Workload, smear: bool):
    q, R, phi0 = kin["q"][:, None], kin["R"][:, None], kin["phi0"][:, None]
    cx, cy = kin["cx"][:, None], kin["cy"][:, None]
    Az = np.nan_to_num(A)
    x, y = _helix_point(cx, cy, R, q, phi0, Az)
    z = kin["z0"][:, None] + R * Az * kin["cot"][:, None]
    barrel = K == 0
    if w.noise_frac > 0.0:
        noise = rng.random(A.shape) < w.noise_frac
        phin = rng.uniform(-np.pi, np.pi, A.shape)
        rb = np.hypot(x, y)
        zb = rng.uniform(-BARREL_HALF_LENGTH, BARREL_HALF_LENGTH, A.shape)
        rd = rng.uniform(BARREL_R_MIN, BARREL_R_MAX, A.shape)
        rn = np.where(barrel, rb, rd)
        x = np.where(noise, rn * np.cos(phin), x)
        y = np.where(noise, rn * np.sin(phin), y)
        z = np.where(noise & barrel, zb, z)
    if smear:
        g1 = rng.normal(0.0, SMEAR_MM, A.shape)
        g2 = rng.normal(0.0, SMEAR_MM, A.shape)
        r = np.hypot(x, y)
        phi = np.arctan2(y, x) + g1 / np.maximum(r, 1e-9)
        xb, yb, zb2 = r * np.cos(phi), r * np.sin(phi), z + g2
        xd, yd = x + g1, y + g2
        x = np.where(barrel, xb, xd)
        y = np.where(barrel, yb, yd)
        z = np.where(barrel, zb2, z)
    return x, y, z


GEN_CHUNK = 65536


def gen_tracks(w: Workload, n_tracks: Optional[int] = None, seed: Optional[int] = None,
               smear: bool = True, pad_value: float = 0.0) -> TrackBatch:
    """Seeded synthetic helix tracks for workload w: hits [B, T, 5] fp32 in
    (x, y, z, r, phi), n_hits [B] int32, pads filled with pad_value.

    Tracks are drawn in chunks of GEN_CHUNK; chunk c uses the stream
    PCG64(SeedSequence([seed, c])), so a batch is the same on every machine and
    its memory use stays bounded."""
    B = w.n_tracks if n_tracks is None else int(n_tracks)
    s0 = w.track_seed if seed is None else seed
    parts = []
    for c, b0 in enumerate(range(0, B, GEN_CHUNK)):
        rng = np.random.Generator(np.random.PCG64(np.random.SeedSequence([s0, c])))
        parts.append(_gen_chunk(w, min(GEN_CHUNK, B - b0), rng, smear, pad_value))
    if len(parts) == 1:
        return parts[0]
    return TrackBatch(hits=np.concatenate([p.hits for p in parts]),
                      n_hits=np.concatenate([p.n_hits for p in parts]),
                      kind=np.concatenate([p.kind for p in parts]),
                      truth=np.concatenate([p.truth for p in parts]),
                      kin={k: np.concatenate([p.kin[k] for p in parts]) for k in parts[0].kin})


def _gen_chunk(w: Workload, B: int, rng, smear: bool, pad_value: float) -> TrackBatch:
    T = w.model.max_hits
    max_keep = MAX_TRACK_HITS if w.layout == "barrel_endcap" else T

    kin_all: Dict[str, List[np.ndarray]] = {}
    A_rows, K_rows = [], []
    need = B
    for _ in range(64):
        if need == 0:
            break
        n_draw = need if w.layout != "barrel_endcap" else int(need * 1.3) + 16
        kin, A, K = _gen_raw(rng, n_draw, w)
        cnt = np.sum(~np.isnan(A), axis=1)
        keep = np.nonzero(cnt >= w.min_hits)[0][:need]
        for k, v in kin.items():
            kin_all.setdefault(k, []).append(v[keep])
        A_rows.append(A[keep])
        K_rows.append(K[keep])
        need -= keep.size
    if need:
        raise RuntimeError("track generator could not draw enough tracks")
    S = max(a.shape[1] for a in A_rows)
    A = np.concatenate([np.pad(a, ((0, 0), (0, S - a.shape[1])), constant_values=np.nan) for a in A_rows])
    K = np.concatenate([np.pad(k, ((0, 0), (0, S - k.shape[1]))) for k in K_rows])
    kin = {k: np.concatenate(v) for k, v in kin_all.items()}

    cnt = np.minimum(np.sum(~np.isnan(A), axis=1), max_keep)
    A = A[:, :max_keep]
    K = K[:, :max_keep]
    if w.drop_max > 0:
        # drop k ~ U{0..drop_max} hits at uniformly chosen positions (order kept)
        k_drop = rng.integers(0, w.drop_max + 1, B)
        keys = rng.random(A.shape)
        keys = np.where(np.arange(A.shape[1])[None, :] < cnt[:, None], keys, np.inf)
        rank = np.argsort(np.argsort(keys, axis=1), axis=1)
        dropped = rank < k_drop[:, None]
        A = np.where(dropped, np.nan, A)
        order = np.argsort(np.where(np.isnan(A), np.inf, A), axis=1, kind="stable")
        A = np.take_along_axis(A, order, axis=1)
        K = np.take_along_axis(K, order, axis=1)
        cnt = cnt - k_drop
    x, y, z = _positions(kin, A, K, rng, w, smear)
    r = np.hypot(x, y)
    phi = np.arctan2(y, x)
    feats = np.stack([x, y, z, r, phi], axis=-1)        # [B, S, 5] fp64
    hits = np.full((B, T, N_FEATURES), pad_value, dtype=np.float32)
    S2 = min(T, feats.shape[1])
    valid = np.arange(S2)[None, :] < cnt[:, None]
    hits[:, :S2, :] = np.where(valid[..., None], feats[:, :S2, :].astype(np.float32), np.float32(pad_value))
    p = kin["pt"] / np.sin(kin["theta"])
    truth = np.stack([kin["d0"], kin["z0"], kin["phi0"], kin["theta"], kin["q"] / p], axis=1)
    kind = np.full((B, T), -1, dtype=np.int8)
    kind[:, :S2] = np.where(valid, K[:, :S2], -1)
    return TrackBatch(hits=hits, n_hits=cnt.astype(np.int32), kind=kind, truth=truth, kin=kin)


def paper_hits(tb: TrackBatch, w: Workload) -> np.ndarray:
    """The 15-feature hit rows of the paper's model (PAPER_FEATURES) for a batch:
    the 12 measured features derived from the stored fp32 (x, y, z, r, phi) in
    fp64 and rounded to fp32; the three seed features left zero (the seed fills
    them, on the device in place); padding rows zero.  Surface index: the nearest
    barrel radius, or the nearest disk |z| (noise hits stay on their surface)."""
    h = tb.hits.astype(np.float64)
    x, y, z, r, phi = (h[..., k] for k in range(5))
    valid = tb.kind >= 0
    radii = np.linspace(BARREL_R_MIN, BARREL_R_MAX, w.n_barrel if w.layout == "sweep" else 10)
    bi = np.argmin(np.abs(r[..., None] - radii), axis=-1)
    di = np.argmin(np.abs(np.abs(z)[..., None] - np.asarray(DISK_Z)), axis=-1)
    with np.errstate(divide="ignore", invalid="ignore"):
        eta = np.arcsinh(z / np.where(r > 0, r, 1.0))
    cols = [x, y, z, r, phi, np.arctan2(r, z), eta, np.hypot(r, z), np.cos(phi), np.sin(phi),
            tb.kind.astype(np.float64), np.where(tb.kind == 1, di, bi).astype(np.float64)]
    out = np.zeros(h.shape[:2] + (15,), dtype=np.float32)
    out[..., :12] = np.where(valid[..., None], np.stack(cols, axis=-1), 0.0).astype(np.float32)
    return out


def length_histogram(n_hits: np.ndarray) -> Dict[int, int]:
    v, c = np.unique(n_hits, return_counts=True)
    return {int(a): int(b) for a, b in zip(v, c)}
