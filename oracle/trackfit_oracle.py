"""CPU oracle for the bidirectional minGRU track-fit encoder (inference only).

TEST INFRASTRUCTURE.  Only the tests, the smoke check and the bench's CPU
baseline leg may import this module.  It shares no code with the CUDA path and
imports nothing from the library package: its inputs (configuration numbers,
weight blob, hits, hit counts) are handed to it as plain arrays.

Everything is computed in fp64 with plain numpy: elementwise formulas and
matmul as the only library step.  Each function states the passage of the paper
it follows ("Fast and Precise Learned Charged-Particle Trajectory Regression at
the LHC").  Where the paper is silent, the reading taken is stated in the
function that takes it.

Reduced-precision modes (precision = 1: bf16, precision = 2: fp16): the paper
runs the encoder GEMMs in fp16 with fp32 recurrence state (Sec. 3.5).  The oracle
then rounds exactly the operands of the per-hit GEMMs to that format (round to
nearest even, from fp64): the Fourier vector, the embedding hidden activation,
the pre-normed layer input, the concatenated scan states, the gated residual x',
the MLP hidden activation, and the weights of those GEMMs.  Everything else
(biases, gates, scan state, residual stream, pooling, head) stays fp64.

Parity status: agreement with the paper's trained model is unpinned (no trained
weights, data or printed activations exist); the functions here are pinned by
closed forms, invariants and brute force in tests/test_oracle_*.py.
"""
from __future__ import annotations

from typing import Dict, Optional

import numpy as np

__all__ = ["bf16_round", "fp16_round", "sigmoid", "silu", "rmsnorm", "normalise", "fourier", "linear_scan",
           "mingru_layer_scans", "embed", "encoder_layer", "encoder_layer_concat", "attention",
           "encoder_layer_attention", "pool", "head", "forward",
           "split_blob"]


# ---------------------------------------------------------------------------
# elementary functions
# ---------------------------------------------------------------------------

def bf16_round(x: np.ndarray) -> np.ndarray:
    """Round fp64 values to the nearest bf16 value (ties to even); result in fp64.

    bf16 keeps fp32's 8 exponent bits and 7 mantissa bits.  For normal numbers
    this keeps the top 7 of fp64's 52 mantissa bits; below 2^-126 bf16 is
    subnormal with a fixed spacing of 2^-133.  NaN and inf pass through."""
    x = np.asarray(x, dtype=np.float64)
    bits = x.view(np.uint64)
    drop = np.uint64(52 - 7)
    lsb = (bits >> drop) & np.uint64(1)
    half = np.uint64((1 << (52 - 7 - 1)) - 1)
    rounded = ((bits + half + lsb) >> drop) << drop
    out = rounded.view(np.float64)
    tiny = np.abs(x) < 2.0 ** -126
    step = 2.0 ** -133
    out = np.where(tiny, np.round(np.where(tiny, x, 0.0) / step) * step, out)
    out = np.where(np.isfinite(x), out, x)
    # values past the largest bf16 round to inf
    return out


def fp16_round(x: np.ndarray) -> np.ndarray:
    """Round fp64 values to the nearest IEEE binary16 value (ties to even); result
    in fp64.  numpy converts float64 to float16 directly with that rounding."""
    with np.errstate(over="ignore"):
        return np.asarray(x, dtype=np.float64).astype(np.float16).astype(np.float64)


def sigmoid(x):
    """Logistic function 1 / (1 + exp(-x)): the minGRU gate sigma (Sec. 3.2)."""
    with np.errstate(over="ignore"):
        return 1.0 / (1.0 + np.exp(-x))


def silu(x):
    """x * sigmoid(x).  The paper does not name its activations; SiLU is the reading."""
    return x * sigmoid(x)


def rmsnorm(x, g, eps):
    """Root-mean-square normalisation over the last axis with gain g (Zhang and
    Sennrich 2019; the paper normalises the pooled vector before the head, Sec. 3.2)."""
    ms = np.mean(x * x, axis=-1, keepdims=True)
    return x / np.sqrt(ms + eps) * g


# ---------------------------------------------------------------------------
# hit features (Sec. 3.2: min-max normalisation, 16-scale Fourier featurisation)
# ---------------------------------------------------------------------------

def normalise(hits, feat_min, feat_max):
    """Min-max normalise every feature to [0, 1] with fixed constants (Sec. 3.2)."""
    lo = np.asarray(feat_min, dtype=np.float64)
    hi = np.asarray(feat_max, dtype=np.float64)
    return (np.asarray(hits, dtype=np.float64) - lo) / (hi - lo)


def fourier(u, scales):
    """Multi-scale Fourier features of Sec. 3.2 (after Tancik et al.).

    For feature f and scale s_k the pair (sin(pi s_k u_f), cos(pi s_k u_f)) is
    emitted.  Layout per hit: for each feature f the K sines, then the K cosines,
    so the vector has 2*F*K entries (the paper's 15*16*2 = 480; 5*16*2 = 160 here)."""
    s = np.asarray(scales, dtype=np.float64)
    arg = np.pi * u[..., :, None] * s                    # [..., F, K]
    e = np.concatenate([np.sin(arg), np.cos(arg)], axis=-1)   # [..., F, 2K]
    return e.reshape(u.shape[:-1] + (2 * u.shape[-1] * s.size,))


# ---------------------------------------------------------------------------
# recurrence (Sec. 3.2, Eq. 2)
# ---------------------------------------------------------------------------

def linear_scan(a, b, x, valid, reverse=False):
    """Masked gated linear recurrence h_t = a_t * h_{t-1} + b_t * x_t along axis 1.

    a, b, x: [B, T, C]; valid: [B, T] bool.  The state starts at zero.  At an
    invalid step the state is carried unchanged and the output is 0 (selected,
    never multiplied, so NaN in padded inputs cannot leak).  reverse=True runs
    from t = T-1 down to 0, i.e. the reverse direction of Sec. 3.2."""
    B, T, C = x.shape
    h = np.zeros((B, C), dtype=np.float64)
    out = np.zeros((B, T, C), dtype=np.float64)
    steps = range(T - 1, -1, -1) if reverse else range(T)
    for t in steps:
        v = valid[:, t, None]
        h = np.where(v, a[:, t] * h + b[:, t] * x[:, t], h)
        out[:, t] = np.where(v, h, 0.0)
    return out


def mingru_layer_scans(z_f, n_f, z_b, n_b, valid):
    """The two scans of one bidirectional minGRU layer (Sec. 3.2).

    Eq. 2 reads h_t = h_{t-1} + z_t * (n_t - h_{t-1}), which is the linear
    recurrence with a_t = 1 - z_t, b_t = z_t, x_t = n_t.  The forward scan runs
    over the hits in time order, the reverse scan in the opposite order; each
    direction has its own gate and candidate."""
    h_f = linear_scan(1.0 - z_f, z_f, n_f, valid, reverse=False)
    h_b = linear_scan(1.0 - z_b, z_b, n_b, valid, reverse=True)
    return h_f, h_b


# ---------------------------------------------------------------------------
# network blocks
# ---------------------------------------------------------------------------

def _op(x, prec):
    """Operand of a per-hit GEMM: rounded to bf16 (prec 1) or fp16 (prec 2), else unchanged."""
    if prec == 1:
        return bf16_round(x)
    if prec == 2:
        return fp16_round(x)
    return x


def _lin(x, w, b, prec):
    """y = x W^T + b with W in PyTorch [out][in] order; GEMM operands rounded per prec."""
    return _op(x, prec) @ _op(np.asarray(w, dtype=np.float64), prec).T + b


def embed(e, W, bf16):
    """Dense network from the Fourier vector to d_model (Sec. 3.2).  The paper does
    not give its depth; reading: two layers with SiLU, x0 = W2 SiLU(W1 e + b1) + b2."""
    hdn = silu(_lin(e, W["emb.w1"], W["emb.b1"], bf16))
    return _lin(hdn, W["emb.w2"], W["emb.b2"], bf16)


def encoder_layer(x, W, l, cfg, valid, bf16, last_endpoints=False):
    """One bidirectional minGRU layer (Sec. 3.2) in the merged form used here.

    1. x_hat = RMSNorm(x) * g                                  (pre-norm; reading)
    2. [p_zf, n_f, p_zb, n_b, p_g] = W_in x_hat + b_in         (Sec. 3.2: gates and
       candidates are linear in the layer input, z = sigma(Linear), n = Linear)
    3. forward and reverse scans of Eq. 2 under the padding mask
    4. x' = x + (W_m [h_f; h_b] + b_m) * sigma(p_g)            (merge with output gate)
    5. x_next = x' + W_2 SiLU(W_1 x' + b_1) + b_2, padded hits set to 0   (MLP)
    Steps 4-5 read the two directions through a gated merge and an MLP instead of the
    paper's plain concatenation; the concatenation is the special case the tests pin.
    Returns (x_next, h_f, h_b); with last_endpoints the merge and MLP are skipped."""
    D, H = cfg["d_model"], cfg["d_hidden"]
    p = f"layer{l}."
    xh = rmsnorm(x, W[p + "g"], cfg["rms_eps"])
    proj = _lin(xh, W[p + "w_in"], W[p + "b_in"], bf16)
    z_f = sigmoid(proj[..., 0:H])
    n_f = proj[..., H:2 * H]
    z_b = sigmoid(proj[..., 2 * H:3 * H])
    n_b = proj[..., 3 * H:4 * H]
    gate = sigmoid(proj[..., 4 * H:4 * H + D])
    h_f, h_b = mingru_layer_scans(z_f, n_f, z_b, n_b, valid)
    if last_endpoints:
        return x, h_f, h_b
    y = np.concatenate([h_f, h_b], axis=-1)
    m = _lin(y, W[p + "w_m"], W[p + "b_m"], bf16)
    x1 = x + m * gate
    u = silu(_lin(x1, W[p + "w1"], W[p + "b1"], bf16))
    x2 = x1 + _lin(u, W[p + "w2"], W[p + "b2"], bf16)
    return np.where(valid[..., None], x2, 0.0), h_f, h_b


def encoder_layer_concat(x, W, l, cfg, valid, prec):
    """One layer of the paper's own topology (Sec. 3.2): the layer input is
    projected linearly to the forward and reverse gates and candidates
    [p_zf, n_f, p_zb, n_b] = W_in x + b_in (z = sigma(p_z)), the forward and
    reverse scans of Eq. 2 run under the padding mask, and the two directions'
    states are concatenated (2H wide) into the next layer.  The paper names no
    normalisation inside the encoder; none is applied.  Returns (y, h_f, h_b),
    y = [h_f; h_b], zero on padded hits (the scans output 0 there)."""
    H = cfg["d_hidden"]
    p = f"layer{l}."
    proj = _lin(x, W[p + "w_in"], W[p + "b_in"], prec)
    z_f = sigmoid(proj[..., 0:H])
    n_f = proj[..., H:2 * H]
    z_b = sigmoid(proj[..., 2 * H:3 * H])
    n_b = proj[..., 3 * H:4 * H]
    h_f, h_b = mingru_layer_scans(z_f, n_f, z_b, n_b, valid)
    return np.concatenate([h_f, h_b], axis=-1), h_f, h_b


def attention(q, k, v, valid, n_heads):
    """Multi-head self-attention within each track (Vaswani et al. 2017), the
    token mixing of the paper's Transformer encoder (App. A.3, Tab. A.1: full
    attention over a track's hits).  q, k, v: [B, T, D], split into n_heads heads
    of D / n_heads channels; per head the weights are the softmax over the track's
    valid hits of q . k / sqrt(D / n_heads) and the output their weighted sum of v.
    Padded hits are no keys (their weight is exactly 0); a padded query's output
    is 0."""
    B, T, D = q.shape
    dh = D // n_heads
    qh, kh, vh = (np.asarray(a, dtype=np.float64).reshape(B, T, n_heads, dh) for a in (q, k, v))
    sc = np.einsum("bthd,bshd->bhts", qh, kh) / np.sqrt(dh)
    sc = np.where(valid[:, None, None, :], sc, -np.inf)
    sc = sc - np.max(sc, axis=-1, keepdims=True)      # the softmax is unchanged by the shift
    w = np.exp(sc)
    w = w / np.sum(w, axis=-1, keepdims=True)
    o = np.einsum("bhts,bshd->bthd", w, vh).reshape(B, T, D)
    return np.where(valid[..., None], o, 0.0)


def encoder_layer_attention(x, W, l, cfg, valid, prec):
    """One layer of the Transformer encoder (reading; the paper names only a
    general-purpose Transformer of the same parameter count, App. A.3): pre-norm
    attention and MLP blocks with residuals (MLP hidden width d_hidden),
      x' = x + W_o attention(W_qkv RMSNorm(x) g_1 + b_qkv) + b_o
      x_next = x' + W_2 SiLU(W_1 RMSNorm(x') g_2 + b_1) + b_2,  padded hits set to 0.
    With 16-bit operands the projections' operands are rounded as in the
    recurrent encoder; the attention itself (scores, softmax, weighted sum) is
    full precision.  No positional encoding: the Fourier features of the hit
    positions carry where a hit is."""
    D = cfg["d_model"]
    p = f"layer{l}."
    qkv = _lin(rmsnorm(x, W[p + "g1"], cfg["rms_eps"]), W[p + "w_qkv"], W[p + "b_qkv"], prec)
    o = attention(qkv[..., 0:D], qkv[..., D:2 * D], qkv[..., 2 * D:3 * D], valid, cfg["n_heads"])
    x1 = x + _lin(o, W[p + "w_o"], W[p + "b_o"], prec)
    u = silu(_lin(rmsnorm(x1, W[p + "g2"], cfg["rms_eps"]), W[p + "w1"], W[p + "b1"], prec))
    x2 = x1 + _lin(u, W[p + "w2"], W[p + "b2"], prec)
    return np.where(valid[..., None], x2, 0.0), None, None


def pool(x, h_f, h_b, n_hits, valid, mode):
    """Track readout.  mode 0 (mean): average of the last layer's output over the
    valid hits (masked pooling).  mode 1 (endpoints, Sec. 3.2): the forward state at
    the outermost hit concatenated with the reverse state at the innermost hit."""
    if mode == 0:
        s = np.sum(np.where(valid[..., None], x, 0.0), axis=1)
        return s / n_hits[:, None].astype(np.float64)
    idx = np.arange(x.shape[0])
    return np.concatenate([h_f[idx, n_hits - 1], h_b[:, 0]], axis=-1)


def head(pv, W, cfg):
    """Sec. 3.2-3.3: RMSNorm, two-layer head (hidden 128) to 5 x 7 quantiles; the
    median quantile (index 3 of 7, parameter-major layout) is the point estimate.
    Kept in full precision in both modes."""
    hn = rmsnorm(pv, W["head.g"], cfg["rms_eps"])
    hid = silu(hn @ np.asarray(W["head.w1"], np.float64).T + W["head.b1"])
    q = hid @ np.asarray(W["head.w2"], np.float64).T + W["head.b2"]
    nq = cfg["n_quantiles"]
    q = q.reshape(q.shape[0], q.shape[1] // nq, nq)
    return q[:, :, nq // 2], q


# ---------------------------------------------------------------------------
# whole forward
# ---------------------------------------------------------------------------

def _layout(cfg):
    D, H, E = cfg["d_model"], cfg["d_hidden"], 2 * cfg["n_features"] * cfg["n_fourier"]
    P = D if cfg["pool"] == 0 else 2 * H
    Hh, Q = cfg["head_hidden"], 5 * cfg["n_quantiles"]
    lay = [("emb.w1", (D, E)), ("emb.b1", (D,)), ("emb.w2", (D, D)), ("emb.b2", (D,))]
    concat = int(cfg.get("topology", 0)) == 1
    attn = int(cfg.get("topology", 0)) == 2
    if concat:
        P = 2 * H
    if attn:
        P = D
    for l in range(cfg["n_layers"]):
        p = f"layer{l}."
        if attn:
            lay += [(p + "g1", (D,)), (p + "w_qkv", (3 * D, D)), (p + "b_qkv", (3 * D,)), (p + "w_o", (D, D)),
                    (p + "b_o", (D,)), (p + "g2", (D,)), (p + "w1", (H, D)), (p + "b1", (H,)),
                    (p + "w2", (D, H)), (p + "b2", (D,))]
            continue
        if concat:   # Sec. 3.2: W_in from the layer input (D, then 2H) to the gates and candidates
            I = D if l == 0 else 2 * H
            lay += [(p + "w_in", (4 * H, I)), (p + "b_in", (4 * H,))]
            continue
        lay += [(p + "g", (D,)), (p + "w_in", (4 * H + D, D)), (p + "b_in", (4 * H + D,)),
                (p + "w_m", (D, 2 * H)), (p + "b_m", (D,)), (p + "w1", (D, D)), (p + "b1", (D,)),
                (p + "w2", (D, D)), (p + "b2", (D,))]
    lay += [("head.g", (P,)), ("head.w1", (Hh, P)), ("head.b1", (Hh,)), ("head.w2", (Q, Hh)),
            ("head.b2", (Q,))]
    return lay


def split_blob(cfg, blob) -> Dict[str, np.ndarray]:
    """Name the tensors of the flat fp32 weight blob (order documented in
    include/trackfit.h), converted to fp64."""
    blob = np.asarray(blob)
    out, off = {}, 0
    for name, shape in _layout(cfg):
        n = int(np.prod(shape))
        out[name] = blob[off:off + n].astype(np.float64).reshape(shape)
        off += n
    if off != blob.size:
        raise ValueError(f"weight blob has {blob.size} values, expected {off}")
    return out


def forward(cfg: dict, blob, hits, n_hits, capture: Optional[dict] = None):
    """Track parameters (d0, z0, phi, theta, q/p) for every track: [B, 5] fp64.

    cfg: dict with d_model, d_hidden, n_layers, n_features, n_fourier, head_hidden,
    n_quantiles, precision (0 fp32, 1 bf16 operands, 2 fp16 operands), pool (0 mean, 1 endpoints),
    feat_min, feat_max, fourier_scale, rms_eps, and topology (0: the gated merge
    and MLP of encoder_layer, the default; 1: the paper's concatenation,
    encoder_layer_concat; 2: the Transformer encoder, encoder_layer_attention, with
    n_heads, mean pooling only).  hits: [B, T, n_features]; n_hits: [B].
    Tracks whose hit count is outside [1, T] give a NaN row.  The output is the
    median quantile of the head directly (no seed decode)."""
    W = split_blob(cfg, blob)
    bf16 = int(cfg["precision"])      # operand rounding: 0 none, 1 bf16, 2 fp16
    hits = np.asarray(hits)
    n_hits = np.asarray(n_hits).astype(np.int64)
    B, T, _ = hits.shape
    bad = (n_hits < 1) | (n_hits > T)
    n_ok = np.where(bad, 1, n_hits)
    valid = np.arange(T)[None, :] < n_ok[:, None]
    u = normalise(hits, cfg["feat_min"], cfg["feat_max"])
    e = fourier(u, cfg["fourier_scale"])
    x = np.where(valid[..., None], embed(e, W, bf16), 0.0)
    L = cfg["n_layers"]
    endpoints = int(cfg["pool"]) == 1
    h_f = h_b = None
    for l in range(L):
        if int(cfg.get("topology", 0)) == 1:
            x, h_f, h_b = encoder_layer_concat(x, W, l, cfg, valid, bf16)
        elif int(cfg.get("topology", 0)) == 2:
            x, h_f, h_b = encoder_layer_attention(x, W, l, cfg, valid, bf16)
        else:
            x, h_f, h_b = encoder_layer(x, W, l, cfg, valid, bf16, last_endpoints=endpoints and l == L - 1)
    pv = pool(x, h_f, h_b, n_ok, valid, int(cfg["pool"]))
    out, q = head(pv, W, cfg)
    out = np.where(bad[:, None], np.nan, out)
    if capture is not None:
        capture.update(pooled=pv, quantiles=q, x_last=x)
    return out
