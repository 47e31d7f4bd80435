"""Pins for the oracle's Transformer encoder (App. A.3, Tab. A.1), no GPU: the
attention against a brute-force loop over heads, queries and keys written with
scalar exponentials; the closed form with zero queries (every weight 1/n, the
output the mean of the track's values); a one-hit track (its own value); the
layer against its two residual blocks written out with saturated projections;
hit-order equivariance (no positional encoding: permuting a track's hits
permutes its outputs and leaves the mean-pooled readout unchanged); NaN pads and
batch splits; and the parameter count of the workload."""
import dataclasses
import math

import numpy as np
import pytest

from oracle import trackfit_oracle as O
from paper_2609_32479_gb300 import workloads as Wl


def attn_model(T=7, D=8, H=12, L=2, heads=2, F=5, **kw):
    fm = tuple(Wl.FEAT_MIN) + (-1.0,) * (F - 5)
    fx = tuple(Wl.FEAT_MAX) + (1.0,) * (F - 5)
    return Wl.ModelConfig(max_hits=T, d_model=D, d_hidden=H, n_layers=L, n_features=F, n_heads=heads,
                          topology=Wl.TOPOLOGY_ATTENTION, feat_min=fm[:F], feat_max=fx[:F], **kw)


def tracks(model, B, seed=5):
    tb = Wl.gen_tracks(Wl.Workload("t", B, model.with_(n_features=5, feat_min=Wl.FEAT_MIN, feat_max=Wl.FEAT_MAX,
                                                       topology=Wl.TOPOLOGY_MERGE), min_hits=1), seed=seed)
    n = np.random.default_rng(seed).integers(1, model.max_hits + 1, B).astype(np.int32)
    hits = tb.hits
    if model.n_features > 5:
        extra = np.random.default_rng(seed + 1).uniform(-1, 1, hits.shape[:2] + (model.n_features - 5,))
        hits = np.concatenate([hits, extra.astype(np.float32)], axis=-1)
    return hits, n


def brute_attention(q, k, v, n, heads):
    """Scalar loops: for each track, head and valid query, softmax over the valid
    keys of the scaled dot products, weighted sum of the values."""
    B, T, D = q.shape
    dh = D // heads
    out = np.zeros((B, T, D))
    for b in range(B):
        for h in range(heads):
            c = slice(h * dh, (h + 1) * dh)
            for t in range(n[b]):
                s = [sum(q[b, t, c][i] * k[b, j, c][i] for i in range(dh)) / math.sqrt(dh) for j in range(n[b])]
                m = max(s)
                e = [math.exp(x - m) for x in s]
                z = sum(e)
                for j in range(n[b]):
                    out[b, t, c] += e[j] / z * v[b, j, c]
    return out


def test_attention_matches_brute_force():
    g = np.random.default_rng(3)
    B, T, D, heads = 5, 6, 8, 2
    q, k, v = (g.normal(0.0, 1.5, (B, T, D)) for _ in range(3))
    n = np.array([1, 6, 3, 5, 2])
    valid = np.arange(T)[None, :] < n[:, None]
    got = O.attention(q, k, v, valid, heads)
    np.testing.assert_allclose(got, brute_attention(q, k, v, n, heads), rtol=1e-12, atol=1e-13)
    assert np.all(got[~valid] == 0.0)


def test_zero_queries_average_the_values_and_one_hit_returns_its_value():
    g = np.random.default_rng(4)
    B, T, D = 6, 9, 12
    k, v = g.normal(size=(B, T, D)), g.normal(size=(B, T, D))
    n = np.array([1, 2, 9, 4, 7, 1])
    valid = np.arange(T)[None, :] < n[:, None]
    got = O.attention(np.zeros((B, T, D)), k, v, valid, 3)
    for b in range(B):
        mean = v[b, :n[b]].mean(axis=0)
        np.testing.assert_allclose(got[b, :n[b]], np.broadcast_to(mean, (n[b], D)), rtol=1e-13, atol=1e-14)
    one = n == 1
    np.testing.assert_allclose(O.attention(g.normal(size=(B, T, D)), k, v, valid, 3)[one, 0], v[one, 0], rtol=1e-14)


def test_layer_with_zero_queries_is_its_two_residual_blocks():
    """W_q = 0, b_q = 0: the attention block adds W_o mean_s(v_s) + b_o to every
    valid hit (v = W_v RMSNorm(x) g_1 + b_v); the MLP block adds W_2 SiLU(W_1
    RMSNorm(x') g_2 + b_1) + b_2.  Written out per track."""
    m = attn_model(L=1)
    D = m.d_model
    hits, n = tracks(m, 8)
    blob = Wl.gen_weights(m, 9)
    W = Wl.split_weights(m, blob.copy())
    W["layer0.w_qkv"][0:D] = 0.0
    W["layer0.b_qkv"][0:D] = 0.0
    W["layer0.g1"][:] = np.linspace(0.5, 1.5, D)
    blob2 = Wl.join_weights(m, W)
    cfg = dataclasses.asdict(m)
    Wd = O.split_blob(cfg, blob2)
    cap = {}
    O.forward(cfg, blob2, hits, n, capture=cap)
    e = O.fourier(O.normalise(hits, m.feat_min, m.feat_max), m.fourier_scale)
    x = O.embed(e, Wd, 0)

    def rms(a, gain):
        return a / np.sqrt(np.mean(a * a, axis=-1, keepdims=True) + m.rms_eps) * gain

    for b in range(len(n)):
        xb = x[b, :n[b]]
        vb = rms(xb, Wd["layer0.g1"]) @ Wd["layer0.w_qkv"][2 * D:].T + Wd["layer0.b_qkv"][2 * D:]
        x1 = xb + vb.mean(axis=0) @ Wd["layer0.w_o"].T + Wd["layer0.b_o"]
        hdn = rms(x1, Wd["layer0.g2"]) @ Wd["layer0.w1"].T + Wd["layer0.b1"]
        x2 = x1 + (hdn / (1.0 + np.exp(-hdn))) @ Wd["layer0.w2"].T + Wd["layer0.b2"]
        np.testing.assert_allclose(cap["x_last"][b, :n[b]], x2, rtol=1e-11, atol=1e-12)
        assert np.all(cap["x_last"][b, n[b]:] == 0.0)
        np.testing.assert_allclose(cap["pooled"][b], x2.mean(axis=0), rtol=1e-11, atol=1e-12)


@pytest.mark.parametrize("prec", [Wl.PRECISION_FP32, Wl.PRECISION_FP16])
def test_hit_order_equivariance(prec):
    """No positional encoding: permuting each track's valid hits permutes the last
    layer's per-hit outputs the same way and leaves the output unchanged."""
    m = attn_model(T=9, L=2, precision=prec)
    hits, n = tracks(m, 10)
    blob = Wl.gen_weights(m, 11)
    cfg = dataclasses.asdict(m)
    cap = {}
    ref = O.forward(cfg, blob, hits, n, capture=cap)
    g = np.random.default_rng(12)
    perm_hits = hits.copy()
    perms = []
    for b in range(len(n)):
        p = g.permutation(n[b])
        perm_hits[b, :n[b]] = hits[b, p]
        perms.append(p)
    cap2 = {}
    got = O.forward(cfg, blob, perm_hits, n, capture=cap2)
    np.testing.assert_allclose(got, ref, rtol=1e-10, atol=1e-12)
    for b in range(len(n)):
        np.testing.assert_allclose(cap2["x_last"][b, :n[b]], cap["x_last"][b, perms[b]], rtol=1e-10, atol=1e-12)


def test_nan_pads_batch_split_and_bad_counts():
    m = attn_model(F=15, heads=4)
    hits, n = tracks(m, 12)
    n[3] = 0
    blob = Wl.gen_weights(m, 4)
    cfg = dataclasses.asdict(m)
    ref = O.forward(cfg, blob, hits, n)
    assert np.all(np.isnan(ref[3])) and np.all(np.isfinite(np.delete(ref, 3, axis=0)))
    nan = hits.copy()
    nan[np.arange(m.max_hits)[None, :] >= n[:, None]] = np.nan
    np.testing.assert_array_equal(O.forward(cfg, blob, nan, n), ref)
    parts = np.concatenate([O.forward(cfg, blob, hits[a:b], n[a:b]) for a, b in ((0, 5), (5, 12))])
    np.testing.assert_allclose(parts, ref, rtol=1e-13, atol=1e-15)


def test_transformer_workload_parameter_count():
    """Embedding 78,080 (as the paper-shaped model); per layer g_1 128 + W_qkv
    384*128 + b_qkv 384 + W_o 128*128 + b_o 128 + g_2 128 + W_1 288*128 + b_1 288 +
    W_2 128*288 + b_2 128 = 140,448, three layers; head on the 128-wide mean:
    128 + 128*128 + 128 + 35*128 + 35 = 21,155."""
    m = Wl.WORKLOADS["transformer"].model
    assert Wl.weight_count(m) == 78080 + 3 * 140448 + 21155
    assert abs(Wl.weight_count(m) / Wl.weight_count(Wl.WORKLOADS["paper"].model) - 1.0) < 0.03
