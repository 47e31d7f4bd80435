"""Pins for the oracle's elementary steps: closed forms, special values, library
routines and brute force on tiny inputs (no GPU)."""
import itertools
import json
import math
import os

import numpy as np
import pytest
import torch

from oracle import trackfit_oracle as O

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")
rng = np.random.default_rng(1234)


# ---------------------------------------------------------------- bf16 rounding

def test_bf16_round_matches_torch_on_fp32_values():
    # fp32 inputs (exact in fp64): direct fp64 -> bf16 rounding must equal torch's
    # fp32 -> bf16 round-to-nearest-even conversion.
    x = np.concatenate([
        rng.standard_normal(20000).astype(np.float32),
        (rng.standard_normal(2000) * 1e-39).astype(np.float32),       # fp32 subnormals
        (rng.standard_normal(2000) * 1e30).astype(np.float32),
        np.array([0.0, -0.0, 1.0, 1.00390625, 1.01171875, -3.0e38], np.float32),
    ])
    # exact ties: mantissa low 16 bits = 0x8000
    ties = (rng.integers(0, 2 ** 15, 1000).astype(np.uint32) << 16) | np.uint32(0x3F808000)
    x = np.concatenate([x, ties.view(np.float32)])
    want = torch.from_numpy(x).to(torch.bfloat16).to(torch.float64).numpy()
    got = O.bf16_round(x.astype(np.float64))
    np.testing.assert_array_equal(got, want)


def test_fp16_round_matches_torch_on_fp32_values():
    x = np.concatenate([rng.standard_normal(20000).astype(np.float32),
                        (rng.standard_normal(2000) * 1e-6).astype(np.float32),     # fp16 subnormals
                        np.array([0.0, 65504.0, 65520.0, 1e6, -1e6, 1.0 + 2.0 ** -11], np.float32)])
    want = torch.from_numpy(x).to(torch.float16).to(torch.float64).numpy()
    np.testing.assert_array_equal(O.fp16_round(x.astype(np.float64)), want)


def test_bf16_round_specials():
    v = np.array([np.inf, -np.inf, np.nan])
    got = O.bf16_round(v)
    assert got[0] == np.inf and got[1] == -np.inf and np.isnan(got[2])


# ---------------------------------------------------------------- activations

def test_sigmoid_silu_special_values():
    assert O.sigmoid(0.0) == 0.5
    assert O.silu(0.0) == 0.0
    x = rng.standard_normal(100) * 5
    np.testing.assert_allclose(O.sigmoid(-x), 1.0 - O.sigmoid(x), rtol=0, atol=1e-15)
    import scipy.special
    np.testing.assert_allclose(O.sigmoid(x), scipy.special.expit(x), rtol=1e-15)
    assert O.sigmoid(-1000.0) == 0.0 and O.sigmoid(1000.0) == 1.0
    # silu(x) -> x for large x, -> 0 for very negative x
    assert abs(O.silu(50.0) - 50.0) < 1e-12 and abs(O.silu(-50.0)) < 1e-18


def test_rmsnorm_closed_forms():
    c, eps = 3.0, 1e-6
    x = np.full((2, 7), c)
    np.testing.assert_allclose(O.rmsnorm(x, 1.0, eps), c / math.sqrt(c * c + eps), rtol=1e-15)
    # unit RMS output without eps; scale invariance; gain applied per channel
    v = rng.standard_normal((4, 9))
    y = O.rmsnorm(v, 1.0, 0.0)
    np.testing.assert_allclose(np.sqrt(np.mean(y * y, -1)), 1.0, rtol=1e-14)
    np.testing.assert_allclose(O.rmsnorm(7.5 * v, 1.0, 0.0), y, rtol=1e-13)
    g = np.arange(1, 10, dtype=np.float64)
    np.testing.assert_allclose(O.rmsnorm(v, g, 0.0), y * g, rtol=1e-14)


# ---------------------------------------------------------------- features

def test_normalise_endpoints():
    lo, hi = (-1.0, 0.0, 10.0), (3.0, 2.0, 30.0)
    h = np.array([[lo, hi, [1.0, 1.0, 20.0]]])
    u = O.normalise(h, lo, hi)
    np.testing.assert_allclose(u[0, 0], 0.0)
    np.testing.assert_allclose(u[0, 1], 1.0)
    np.testing.assert_allclose(u[0, 2], 0.5)


def test_fourier_special_values_and_layout():
    F, K = 5, 16
    s = [2.0 ** (k / 3.0) for k in range(K)]
    e0 = O.fourier(np.zeros((1, F)), s)
    assert e0.shape == (1, 2 * F * K)
    e0 = e0.reshape(F, 2, K)
    np.testing.assert_array_equal(e0[:, 0, :], 0.0)     # sin(0)
    np.testing.assert_array_equal(e0[:, 1, :], 1.0)     # cos(0)
    # u = 1/2 at scale 2: (sin pi, cos pi) = (0, -1); at scale 1: (1, 0)
    e = O.fourier(np.full((1, 1), 0.5), [1.0, 2.0]).reshape(2, 2)
    np.testing.assert_allclose(e, [[1.0, 0.0], [0.0, -1.0]], atol=1e-15)
    # feature-major layout: a nonzero u_f changes only the block of feature f
    for f in range(F):
        u = np.zeros((1, F))
        u[0, f] = 0.3
        blk = O.fourier(u, s).reshape(F, 2, K)
        for g in range(F):
            if g != f:
                np.testing.assert_array_equal(blk[g, 0], 0.0)
                np.testing.assert_array_equal(blk[g, 1], 1.0)
        np.testing.assert_allclose(blk[f, 0], np.sin(np.pi * 0.3 * np.asarray(s)), rtol=1e-15)
        np.testing.assert_allclose(blk[f, 0] ** 2 + blk[f, 1] ** 2, 1.0, rtol=1e-15)


def test_paper_dimension_counts():
    """Sec. 3.2: 15 features x 16 scales give a 480-d vector; 5 x 7 = 35 head outputs."""
    with open(os.path.join(GOLDEN, "paper_dimensions.json")) as fh:
        g = json.load(fh)
    e = O.fourier(np.zeros((1, g["n_features"])), [1.0] * g["n_scales"])
    assert e.shape[-1] == g["fourier_dim"]
    assert g["n_params"] * g["n_quantiles"] == g["head_outputs"]
    assert 2 * g["hidden"] == g["concat_dim"]


# ---------------------------------------------------------------- scan

def _valid(B, T, n=None):
    n = np.full(B, T) if n is None else np.asarray(n)
    return np.arange(T)[None, :] < n[:, None]


def test_scan_prefix_sum():
    x = rng.standard_normal((3, 11, 4))
    one = np.ones_like(x)
    np.testing.assert_allclose(O.linear_scan(one, one, x, _valid(3, 11)), np.cumsum(x, axis=1), rtol=1e-13)
    # reverse: suffix sums
    want = np.flip(np.cumsum(np.flip(x, 1), axis=1), 1)
    np.testing.assert_allclose(O.linear_scan(one, one, x, _valid(3, 11), reverse=True), want, rtol=1e-13)


def test_scan_pointwise_when_a_is_zero():
    b, x = rng.standard_normal((2, 2, 9, 5))
    got = O.linear_scan(np.zeros_like(x), b, x, _valid(2, 9))
    np.testing.assert_array_equal(got, b * x)


def test_scan_geometric_series():
    a, b, c, T = 0.7, 0.4, -1.3, 12
    x = np.full((1, T, 1), c)
    got = O.linear_scan(np.full_like(x, a), np.full_like(x, b), x, _valid(1, T))[0, :, 0]
    t = np.arange(T)
    np.testing.assert_allclose(got, b * c * (1 - a ** (t + 1)) / (1 - a), rtol=1e-14)


@pytest.mark.parametrize("T", [1, 2, 3, 6])
def test_scan_brute_force_unrolled_sum(T):
    a, b, x = rng.uniform(-1.2, 1.2, (3, 2, T, 3))
    got = O.linear_scan(a, b, x, _valid(2, T))
    got_r = O.linear_scan(a, b, x, _valid(2, T), reverse=True)
    for i, t, c in itertools.product(range(2), range(T), range(3)):
        # h_t = sum_{s<=t} (prod_{r=s+1..t} a_r) b_s x_s
        want = sum(np.prod(a[i, s + 1:t + 1, c]) * b[i, s, c] * x[i, s, c] for s in range(t + 1))
        assert abs(got[i, t, c] - want) < 1e-13
        want_r = sum(np.prod(a[i, t:s, c]) * b[i, s, c] * x[i, s, c] for s in range(t, T))
        assert abs(got_r[i, t, c] - want_r) < 1e-13


def test_scan_direction_symmetry():
    a, b, x = rng.uniform(-1, 1, (3, 4, 10, 6))
    fwd = O.linear_scan(a, b, x, _valid(4, 10))
    rev = O.linear_scan(np.flip(a, 1), np.flip(b, 1), np.flip(x, 1), _valid(4, 10), reverse=True)
    np.testing.assert_allclose(np.flip(rev, 1), fwd, rtol=1e-14)


def test_scan_padding_carry_and_nan_pads():
    T, n = 8, np.array([3, 8, 1, 5])
    a, b, x = rng.uniform(-1, 1, (3, 4, T, 2))
    v = _valid(4, T, n)
    xn = np.where(v[..., None], x, np.nan)
    an = np.where(v[..., None], a, np.nan)
    fwd = O.linear_scan(an, b, xn, v)
    rev = O.linear_scan(an, b, xn, v, reverse=True)
    assert np.all(np.isfinite(fwd)) and np.all(np.isfinite(rev))
    for i in range(4):
        m = n[i]
        np.testing.assert_array_equal(fwd[i, m:], 0.0)
        np.testing.assert_array_equal(rev[i, m:], 0.0)
        np.testing.assert_allclose(fwd[i, :m], O.linear_scan(a[i:i + 1, :m], b[i:i + 1, :m], x[i:i + 1, :m],
                                                             _valid(1, m))[0], rtol=1e-15)
        np.testing.assert_allclose(rev[i, :m], O.linear_scan(a[i:i + 1, :m], b[i:i + 1, :m], x[i:i + 1, :m],
                                                             _valid(1, m), reverse=True)[0], rtol=1e-15)


def test_mingru_equation_2_literal():
    """Eq. 2 evaluated literally, h_t = h_{t-1} + z_t (n_t - h_{t-1}), in scalar
    Python, against the oracle's scans."""
    T = 7
    zf, nf, zb, nb = rng.uniform(0, 1, (4, 1, T, 3))
    nf, nb = nf * 4 - 2, nb * 4 - 2
    hf, hb = O.mingru_layer_scans(zf, nf, zb, nb, _valid(1, T))
    for c in range(3):
        h = 0.0
        for t in range(T):
            h = h + zf[0, t, c] * (nf[0, t, c] - h)
            assert abs(hf[0, t, c] - h) < 1e-14
        h = 0.0
        for t in reversed(range(T)):
            h = h + zb[0, t, c] * (nb[0, t, c] - h)
            assert abs(hb[0, t, c] - h) < 1e-14


def test_mingru_gate_extremes():
    T = 6
    n = rng.standard_normal((2, T, 4))
    v = _valid(2, T)
    hf, hb = O.mingru_layer_scans(np.ones_like(n), n, np.ones_like(n), n, v)
    np.testing.assert_array_equal(hf, n)        # z = 1: state is the candidate
    np.testing.assert_array_equal(hb, n)
    hf, hb = O.mingru_layer_scans(np.zeros_like(n), n, np.zeros_like(n), n, v)
    np.testing.assert_array_equal(hf, 0.0)      # z = 0: state stays at h_{-1} = 0
    np.testing.assert_array_equal(hb, 0.0)
