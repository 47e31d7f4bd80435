"""Whole-model pins for the oracle: invariances, closed forms with structured
weights (wiring, operand orientation, layouts) and parameter counts (no GPU)."""
import math

import numpy as np
import pytest

from oracle import trackfit_oracle as O
from paper_2609_32479_gb300 import workloads as Wl
from tests.helpers import cfg_dict

rng = np.random.default_rng(99)


def small_model(T=9, D=8, H=12, L=2, **kw):
    return Wl.ModelConfig(max_hits=T, d_model=D, d_hidden=H, n_layers=L, **kw)


def random_tracks(model, B, n=None, seed=5):
    tb = Wl.gen_tracks(Wl.Workload("t", B, model, min_hits=1), seed=seed)
    hits = tb.hits
    if n is not None:
        n_hits = np.asarray(n, np.int32)
    else:
        n_hits = np.random.default_rng(seed).integers(1, model.max_hits + 1, B).astype(np.int32)
    return hits, n_hits


def zero_weights(model):
    return {name: np.zeros(shape) for name, shape, _ in Wl.weight_layout(model)}


def logit(p):
    return math.log(p / (1 - p))


# ---------------------------------------------------------------- sizes

@pytest.mark.parametrize("name,count", [("tiny", 40259), ("small", 226787), ("medium", 1246371),
                                        ("large", 6458659)])
def test_parameter_counts(name, count):
    m = Wl.workload(name).model
    assert Wl.weight_count(m) == count
    blob = np.zeros(count, np.float32)
    assert sum(v.size for v in O.split_blob(cfg_dict(m), blob).values()) == count


# ---------------------------------------------------------------- invariances

@pytest.mark.parametrize("prec", [0, 1])
def test_padding_invariance_nan_pads(prec):
    m = small_model(precision=prec)
    hits, n = random_tracks(m, 24)
    blob = Wl.gen_weights(m, 3)
    ref = O.forward(cfg_dict(m), blob, hits, n)
    T2 = m.max_hits + 5
    padded = np.full((24, T2, 5), np.nan, np.float32)
    for b in range(24):
        padded[b, :n[b]] = hits[b, :n[b]]
    got = O.forward(cfg_dict(m.with_(max_hits=T2)), blob, padded, n)
    np.testing.assert_allclose(got, ref, rtol=1e-12, atol=1e-14)


def test_track_permutation_and_batch_split():
    m = small_model()
    hits, n = random_tracks(m, 30)
    blob = Wl.gen_weights(m, 4)
    cfg = cfg_dict(m)
    ref = O.forward(cfg, blob, hits, n)
    perm = rng.permutation(30)
    np.testing.assert_allclose(O.forward(cfg, blob, hits[perm], n[perm]), ref[perm], rtol=1e-12, atol=1e-14)
    parts = [O.forward(cfg, blob, hits[a:b], n[a:b]) for a, b in ((0, 7), (7, 8), (8, 30))]
    np.testing.assert_allclose(np.concatenate(parts), ref, rtol=1e-12, atol=1e-14)


def test_reversal_with_direction_swap():
    """Reversing every track's hits while swapping the forward/reverse gate and
    candidate weights and the two column halves of the merge leaves the output
    unchanged under mean pooling (Sec. 3.2 bidirectionality)."""
    m = small_model(T=10, D=6, H=9, L=3)
    H = m.d_hidden
    hits, n = random_tracks(m, 16)
    blob = Wl.gen_weights(m, 7)
    W = Wl.split_weights(m, blob.copy())
    for l in range(m.n_layers):
        p = f"layer{l}."
        for key in ("w_in", "b_in"):
            a = W[p + key].copy()
            W[p + key][0:H], W[p + key][2 * H:3 * H] = a[2 * H:3 * H], a[0:H]
            W[p + key][H:2 * H], W[p + key][3 * H:4 * H] = a[3 * H:4 * H], a[H:2 * H]
        a = W[p + "w_m"].copy()
        W[p + "w_m"][:, 0:H], W[p + "w_m"][:, H:2 * H] = a[:, H:2 * H], a[:, 0:H]
    swapped = Wl.join_weights(m, W)
    rev = hits.copy()
    for b in range(16):
        rev[b, :n[b]] = hits[b, :n[b]][::-1]
    cfg = cfg_dict(m)
    ref = O.forward(cfg, blob, hits, n)
    got = O.forward(cfg, swapped, rev, n)
    np.testing.assert_allclose(got, ref, rtol=1e-11, atol=1e-13)
    # and the unswapped weights do see the reversal (the test is not vacuous)
    assert np.max(np.abs(O.forward(cfg, blob, rev, n) - ref)) > 1e-4


def test_invalid_hit_counts_give_nan_rows_only():
    m = small_model()
    hits, n = random_tracks(m, 6)
    blob = Wl.gen_weights(m, 2)
    cfg = cfg_dict(m)
    ref = O.forward(cfg, blob, hits, n)
    bad = n.copy()
    bad[1], bad[4] = 0, m.max_hits + 1
    got = O.forward(cfg, blob, hits, bad)
    assert np.all(np.isnan(got[[1, 4]]))
    keep = [0, 2, 3, 5]
    np.testing.assert_allclose(got[keep], ref[keep], rtol=1e-12)


# ---------------------------------------------------------------- closed forms

def test_quantile_layout_and_median():
    """Sec. 3.2/3.3: 5 parameters x 7 quantiles, median as point estimate."""
    m = small_model()
    W = zero_weights(m)
    W["head.b2"] = np.arange(35.0)
    hits, n = random_tracks(m, 3)
    out = O.forward(cfg_dict(m), Wl.join_weights(m, W), hits, n)
    np.testing.assert_array_equal(out, np.tile([3.0, 10.0, 17.0, 24.0, 31.0], (3, 1)))


def test_endpoint_readout_geometric_series():
    """Endpoint pooling (Sec. 3.2) with constant gates: the forward state at the last
    hit and the reverse state at the first hit follow the geometric series
    h = n (1 - (1 - z)^{n_hits}); the head then reads them through a permutation."""
    D, H = 2, 3
    m = small_model(T=7, D=D, H=H, L=1, pool=Wl.POOL_ENDPOINTS, head_hidden=6)
    W = zero_weights(m)
    zf, nf = np.array([0.2, 0.5, 0.9]), np.array([1.5, -0.7, 0.3])
    zb, nb = np.array([0.35, 0.8, 0.1]), np.array([-1.1, 0.6, 2.0])
    W["emb.b2"] = np.array([0.5, -0.25])
    W["layer0.b_in"] = np.concatenate([[logit(p) for p in zf], nf, [logit(p) for p in zb], nb, [0.0, 0.0]])
    W["head.g"] = np.ones(6)
    W["head.w1"] = np.roll(np.eye(6), 1, axis=1)          # (W h)_i = h_{(i+1) % 6}
    w2 = np.zeros((35, 6))
    for p in range(5):
        w2[7 * p + 3, p] = 1.0
    W["head.w2"] = w2
    n = np.array([1, 4, 7], np.int32)
    hits, _ = random_tracks(m, 3)
    out = O.forward(cfg_dict(m), Wl.join_weights(m, W), hits, n)
    for i, k in enumerate(n):
        pv = np.concatenate([nf * (1 - (1 - zf) ** k), nb * (1 - (1 - zb) ** k)])
        hn = pv / math.sqrt(np.mean(pv ** 2) + m.rms_eps)
        for p in range(5):
            v = hn[(p + 1) % 6]
            assert abs(out[i, p] - v / (1 + math.exp(-v))) < 1e-6 * abs(v) + 1e-15


def test_merge_column_order_and_gate():
    """The merge reads [h_f; h_b] in that order: a merge row with a single 1 at column
    H + c returns the reverse state of channel c, scaled by the output gate."""
    D, H, T = 3, 4, 6
    m = small_model(T=T, D=D, H=H, L=1)
    W = zero_weights(m)
    W["layer0.g"] = np.ones(D)
    W["layer0.b_in"] = np.concatenate([np.full(H, logit(0.3)), np.full(H, 1.0), np.full(H, logit(0.6)),
                                       np.full(H, -2.0), [logit(0.25), 40.0, 0.0]])
    wm = np.zeros((D, 2 * H))
    wm[0, H + 1] = 1.0         # row 0 <- h_b channel 1
    wm[1, 2] = 1.0             # row 1 <- h_f channel 2
    W["layer0.w_m"] = wm
    x = rng.standard_normal((2, T, D))
    n = np.array([6, 3])
    valid = np.arange(T)[None, :] < n[:, None]
    x = np.where(valid[..., None], x, 0.0)
    x2, _, _ = O.encoder_layer(x, W, 0, cfg_dict(m), valid, False)
    for i in range(2):
        for t in range(n[i]):
            hb = -2.0 * (1 - 0.4 ** (n[i] - t))
            hf = 1.0 * (1 - 0.7 ** (t + 1))
            assert abs(x2[i, t, 0] - (x[i, t, 0] + 0.25 * hb)) < 1e-12
            assert abs(x2[i, t, 1] - (x[i, t, 1] + hf)) < 1e-12
            assert abs(x2[i, t, 2] - x[i, t, 2]) < 1e-15
        assert np.all(x2[i, n[i]:] == 0.0)


def test_mlp_operand_orientation():
    """W_1 and W_2 are [out][in]: W_1 = e_0 e_1^T and W_2 = e_2 e_0^T route
    x'_1 through SiLU into channel 2 and nowhere else."""
    D, H, T = 3, 3, 4
    m = small_model(T=T, D=D, H=H, L=1)
    W = zero_weights(m)
    W["layer0.g"] = np.ones(D)
    W["layer0.w1"] = np.zeros((D, D))
    W["layer0.w1"][0, 1] = 1.0
    W["layer0.w2"] = np.zeros((D, D))
    W["layer0.w2"][2, 0] = 1.0
    W["layer0.b2"] = np.array([0.0, 0.0, 0.125])
    x = rng.standard_normal((1, T, D))
    valid = np.ones((1, T), bool)
    x2, _, _ = O.encoder_layer(x, W, 0, cfg_dict(m), valid, False)
    s = x[..., 1] / (1 + np.exp(-x[..., 1]))
    np.testing.assert_allclose(x2[..., 0], x[..., 0], rtol=0, atol=1e-15)
    np.testing.assert_allclose(x2[..., 1], x[..., 1], rtol=0, atol=1e-15)
    np.testing.assert_allclose(x2[..., 2], x[..., 2] + s + 0.125, rtol=1e-14)


def test_embedding_orientation_and_fourier_index():
    """W_e1[d][j] reads Fourier entry j = f*2K + k (sin) / f*2K + K + k (cos)."""
    m = small_model(T=3, D=3, H=3, L=1)
    K = m.n_fourier
    W = zero_weights(m)
    f, k = 2, 3
    W["emb.w1"][1, f * 2 * K + k] = 1.0          # hidden 1 <- sin(pi s_k u_f)
    W["emb.w1"][2, 4 * 2 * K + K + 0] = 1.0      # hidden 2 <- cos(pi s_0 u_4)
    W["emb.w2"][0, 1] = 1.0
    W["emb.w2"][1, 2] = -1.0
    hits, _ = random_tracks(m, 2)
    u = O.normalise(hits, m.feat_min, m.feat_max)
    e = O.fourier(u, m.fourier_scale)
    x0 = O.embed(e, O.split_blob(cfg_dict(m), Wl.join_weights(m, W)), False)
    a = np.sin(np.pi * m.fourier_scale[k] * u[..., f])
    c = np.cos(np.pi * m.fourier_scale[0] * u[..., 4])
    np.testing.assert_allclose(x0[..., 0], a / (1 + np.exp(-a)), rtol=1e-14, atol=1e-16)
    np.testing.assert_allclose(x0[..., 1], -c / (1 + np.exp(-c)), rtol=1e-14, atol=1e-16)
    np.testing.assert_array_equal(x0[..., 2], 0.0)


def test_mean_pool_divides_by_hit_count():
    """With all matrices zero every valid hit carries the same vector, so the mean
    over valid hits equals it for any hit count (a divisor of T would not)."""
    m = small_model(T=8, D=4, H=6, L=2, head_hidden=4)
    W = zero_weights(m)
    W["emb.b2"] = np.array([0.3, -0.2, 0.7, 0.1])
    for l in range(2):
        W[f"layer{l}.b_in"][4 * 6:] = 40.0     # output gate open
        W[f"layer{l}.b_m"] = np.array([0.05, 0.0, -0.1, 0.2])
        W[f"layer{l}.b2"] = np.array([0.0, 0.01, 0.0, -0.02])
    W["head.g"] = np.ones(4)
    W["head.w1"] = np.eye(4)
    w2 = np.zeros((35, 4))
    for p in range(4):
        w2[7 * p + 3, p] = 1.0
    W["head.w2"] = w2
    hits, _ = random_tracks(m, 3)
    n = np.array([1, 5, 8], np.int32)
    cap = {}
    out = O.forward(cfg_dict(m), Wl.join_weights(m, W), hits, n, capture=cap)
    f = lambda v: np.asarray(v, np.float32).astype(np.float64)     # the blob is fp32
    xL = f(W["emb.b2"]) + 2 * (f(W["layer0.b_m"]) + f(W["layer0.b2"]))
    np.testing.assert_allclose(cap["pooled"], np.tile(xL, (3, 1)), rtol=1e-14)
    hn = xL / math.sqrt(np.mean(xL ** 2) + m.rms_eps)
    np.testing.assert_allclose(out[:, :4], np.tile(hn / (1 + np.exp(-hn)), (3, 1)), rtol=1e-13)


def test_prenorm_makes_the_scans_scale_invariant():
    """The projections read the RMS-normalised input (pre-norm, the reading of
    Sec. 3.2 taken here): scaling a hit's input vector by 8 leaves the gates,
    candidates and so both scans unchanged, up to the eps term (~1e-7 here)."""
    m = small_model(T=7, D=8, H=12, L=1)
    W = O.split_blob(cfg_dict(m), Wl.gen_weights(m, 4))
    x = rng.standard_normal((3, 7, 8))
    valid = np.arange(7)[None, :] < np.array([7, 4, 1])[:, None]
    _, hf1, hb1 = O.encoder_layer(x, W, 0, cfg_dict(m), valid, False)
    _, hf8, hb8 = O.encoder_layer(8.0 * x, W, 0, cfg_dict(m), valid, False)
    np.testing.assert_allclose(hf8, hf1, rtol=1e-5, atol=1e-6)
    np.testing.assert_allclose(hb8, hb1, rtol=1e-5, atol=1e-6)


def test_mlp_reads_the_gated_residual():
    """The MLP acts on x' = x + merge * gate, not on the layer input: with the gate
    open, W_m = 0 and b_m = c, x' = x + c, and with W_1 = W_2 = I the output is
    x' + SiLU(x')."""
    D, H, T = 3, 3, 4
    m = small_model(T=T, D=D, H=H, L=1)
    W = zero_weights(m)
    W["layer0.g"] = np.ones(D)
    W["layer0.b_in"][4 * H:] = 40.0
    c = np.array([0.5, -1.25, 2.0])
    W["layer0.b_m"] = c
    W["layer0.w1"] = np.eye(D)
    W["layer0.w2"] = np.eye(D)
    x = rng.standard_normal((2, T, D))
    valid = np.ones((2, T), bool)
    x2, _, _ = O.encoder_layer(x, W, 0, cfg_dict(m), valid, False)
    x1 = x + c / (1 + math.exp(-40.0))
    np.testing.assert_allclose(x2, x1 + x1 / (1 + np.exp(-x1)), rtol=1e-13, atol=1e-15)


def test_padded_hits_are_zero_in_the_layer_output():
    """Padded hits leave a layer as zero vectors (the layer's last step), whatever
    the biases would put there."""
    m = small_model(T=6, D=8, H=12, L=1)
    W = O.split_blob(cfg_dict(m), Wl.gen_weights(m, 6))
    x = rng.standard_normal((3, 6, 8))
    valid = np.arange(6)[None, :] < np.array([6, 2, 5])[:, None]
    x2, _, _ = O.encoder_layer(x, W, 0, cfg_dict(m), valid, False)
    assert np.all(x2[~valid] == 0.0)
    assert np.all(x2[valid] != 0.0)


def test_mean_pool_reads_valid_hits_only():
    """Masked mean pooling (Sec. 3.2): values in padded rows do not enter the mean."""
    x = rng.standard_normal((3, 5, 4))
    n = np.array([5, 1, 3])
    valid = np.arange(5)[None, :] < n[:, None]
    got = O.pool(x, None, None, n, valid, 0)
    for i in range(3):
        np.testing.assert_allclose(got[i], x[i, :n[i]].mean(axis=0), rtol=1e-14)


def test_bf16_mode_is_close_but_not_identical():
    m = small_model(D=16, H=24)
    hits, n = random_tracks(m, 32)
    blob = Wl.gen_weights(m, 8)
    a = O.forward(cfg_dict(m), blob, hits, n)
    b = O.forward(cfg_dict(m.with_(precision=1)), blob, hits, n)
    rel = np.max(np.abs(a - b)) / np.sqrt(np.mean(a * a))
    assert 1e-5 < rel < 5e-2
