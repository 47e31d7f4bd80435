"""Pins for the oracle's concatenation topology (the paper's own, Sec. 3.2), no GPU:
the parameter count of the paper-shaped model, a closed form with saturated gates
(every state equals its candidate, so each layer is an affine map of its input
and the endpoints are plain matrix products), the reversal symmetry with
direction-swapped weights under both readouts, and NaN-pad invariance."""
import dataclasses

import numpy as np
import pytest

from oracle import trackfit_oracle as O
from paper_2609_32479_gb300 import workloads as Wl


def concat_model(T=9, D=8, H=12, L=2, F=5, pool=Wl.POOL_ENDPOINTS, **kw):
    fm = tuple(Wl.FEAT_MIN) + (-1.0,) * (F - 5)
    fx = tuple(Wl.FEAT_MAX) + (1.0,) * (F - 5)
    return Wl.ModelConfig(max_hits=T, d_model=D, d_hidden=H, n_layers=L, pool=pool, n_features=F,
                          topology=Wl.TOPOLOGY_CONCAT, feat_min=fm[:F], feat_max=fx[:F], **kw)


def tracks(model, B, seed=5):
    tb = Wl.gen_tracks(Wl.Workload("t", B, model.with_(n_features=5, feat_min=Wl.FEAT_MIN, feat_max=Wl.FEAT_MAX),
                                   min_hits=1), seed=seed)
    n = np.random.default_rng(seed).integers(1, model.max_hits + 1, B).astype(np.int32)
    hits = tb.hits
    if model.n_features > 5:
        extra = np.random.default_rng(seed + 1).uniform(-1, 1, hits.shape[:2] + (model.n_features - 5,))
        hits = np.concatenate([hits, extra.astype(np.float32)], axis=-1)
    return hits, n


def test_paper_model_parameter_count():
    """d_model 128, two layers of width 192, 15 features (480 Fourier inputs), 7
    quantiles of 5 parameters: embedding 480*128 + 128 + 128*128 + 128 = 78,080;
    layer 0: 768*128 + 768 = 99,072; layer 1: 768*384 + 768 = 295,680; head on the
    384 endpoint features: 384 + 128*384 + 128 + 35*128 + 35 = 54,179.  (The paper
    states 0.64 M; it does not give the dense network's widths.)"""
    m = Wl.WORKLOADS["paper"].model
    assert Wl.weight_count(m) == 78080 + 99072 + 295680 + 54179
    blob = np.zeros(Wl.weight_count(m), np.float32)
    W = O.split_blob(dataclasses.asdict(m), blob)
    assert W["layer1.w_in"].shape == (768, 384) and W["head.w1"].shape == (128, 384)


@pytest.mark.parametrize("pool", [Wl.POOL_ENDPOINTS, Wl.POOL_MEAN])
def test_saturated_gates_make_each_state_its_candidate(pool):
    """With the update gates at 1 (z = sigma(40) = 1 in fp64) every state is its
    candidate, h_t = n_t: a layer's output is [W_nf y + b_nf; W_nb y + b_nb] of its
    input y, layer 0 reads the embedding and layer 1 the concatenation, and the
    readout takes the forward half at the last hit and the reverse half at the
    first (or the mean over the hits)."""
    m = concat_model(pool=pool)
    D, H = m.d_model, m.d_hidden
    hits, n = tracks(m, 20)
    blob = Wl.gen_weights(m, 3)
    W = Wl.split_weights(m, blob.copy())
    for l in range(m.n_layers):
        p = f"layer{l}."
        for blk in (0, 2):                                 # z_f and z_b rows
            W[p + "w_in"][blk * H:(blk + 1) * H] = 0.0
            W[p + "b_in"][blk * H:(blk + 1) * H] = 40.0
    blob2 = Wl.join_weights(m, W)
    cfg = dataclasses.asdict(m)
    cap = {}
    O.forward(cfg, blob2, hits, n, capture=cap)
    Wd = O.split_blob(cfg, blob2)
    valid = np.arange(m.max_hits)[None, :] < n[:, None]
    e = O.fourier(O.normalise(hits, m.feat_min, m.feat_max), m.fourier_scale)
    y = O.embed(e, Wd, 0)
    for l in range(m.n_layers):
        w, b = Wd[f"layer{l}.w_in"], Wd[f"layer{l}.b_in"]
        y = np.concatenate([y @ w[H:2 * H].T + b[H:2 * H], y @ w[3 * H:4 * H].T + b[3 * H:4 * H]], axis=-1)
        y = np.where(valid[..., None], y, 0.0)
    idx = np.arange(len(n))
    if pool == Wl.POOL_ENDPOINTS:
        want = np.concatenate([y[idx, n - 1, :H], y[:, 0, H:]], axis=-1)
    else:
        want = y.sum(axis=1) / n[:, None]
    np.testing.assert_allclose(cap["pooled"], want, rtol=1e-12, atol=1e-12)
    assert cap["pooled"].shape == (len(n), 2 * H)


@pytest.mark.parametrize("pool", [Wl.POOL_ENDPOINTS, Wl.POOL_MEAN])
def test_reversal_with_direction_swap(pool):
    """Reversing every track's hits while swapping the forward and reverse rows of
    every layer's projection, the two column halves of the projections that read a
    concatenation (layers after the first), and the two halves of the head's input
    leaves the output unchanged (Sec. 3.2: the bidirectional layer and the
    endpoint readout are symmetric)."""
    m = concat_model(T=10, D=6, H=9, L=3, pool=pool)
    H = m.d_hidden
    hits, n = tracks(m, 16)
    blob = Wl.gen_weights(m, 7)
    W = Wl.split_weights(m, blob.copy())
    for l in range(m.n_layers):
        p = f"layer{l}."
        for key in ("w_in", "b_in"):
            a = W[p + key].copy()
            W[p + key][0:2 * H], W[p + key][2 * H:4 * H] = a[2 * H:4 * H], a[0:2 * H]
        if l > 0:
            a = W[p + "w_in"].copy()
            W[p + "w_in"][:, 0:H], W[p + "w_in"][:, H:2 * H] = a[:, H:2 * H], a[:, 0:H]
    for key, axis in (("head.g", 0), ("head.w1", 1)):
        a = W[key].copy()
        sl = (slice(None),) * axis
        W[key][sl + (slice(0, H),)], W[key][sl + (slice(H, 2 * H),)] = a[sl + (slice(H, 2 * H),)], a[sl + (slice(0, H),)]
    swapped = Wl.join_weights(m, W)
    rev = hits.copy()
    for b in range(16):
        rev[b, :n[b]] = hits[b, :n[b]][::-1]
    cfg = dataclasses.asdict(m)
    ref = O.forward(cfg, blob, hits, n)
    np.testing.assert_allclose(O.forward(cfg, swapped, rev, n), ref, rtol=1e-11, atol=1e-13)
    assert np.max(np.abs(O.forward(cfg, blob, rev, n) - ref)) > 1e-4


def test_nan_pads_and_more_features():
    """15 features (the paper's count) and NaN in every padded entry: the output
    equals the run with zero pads, and a batch split changes nothing."""
    m = concat_model(F=15)
    hits, n = tracks(m, 12)
    blob = Wl.gen_weights(m, 4)
    cfg = dataclasses.asdict(m)
    ref = O.forward(cfg, blob, hits, n)
    nan = hits.copy()
    nan[np.arange(m.max_hits)[None, :] >= n[:, None]] = np.nan
    np.testing.assert_allclose(O.forward(cfg, blob, nan, n), ref, rtol=1e-13, atol=1e-15)
    parts = np.concatenate([O.forward(cfg, blob, hits[a:b], n[a:b]) for a, b in ((0, 5), (5, 12))])
    np.testing.assert_allclose(parts, ref, rtol=1e-13, atol=1e-15)
