"""The Transformer encoder of the paper's encoder comparison (App. A.3, Tab. A.1) on
the GPU against the oracle: the paper's 15 features (the seed's three computed by
the seed oracle), d_model 128, three layers of 4-head attention over each track's
hits and an MLP of width 288, mean pooled, in fp32 and with fp16 operands; a
long-track configuration whose attention CTA needs more than 48 KB of shared
memory; the masking, batch-order and packed-input invariances bit-exactly; the
quantile and pooled exports."""
import dataclasses

import numpy as np
import pytest

from oracle import seed_oracle as S
from oracle import trackfit_oracle as O
from paper_2609_32479_gb300 import workloads as W
from tests.helpers import parity_ok

pytestmark = pytest.mark.gpu
torch = pytest.importorskip("torch")


@pytest.fixture(scope="module")
def T():
    import os
    from paper_2609_32479_gb300 import trackfit
    if not os.path.exists(trackfit.LIB_PATH):
        import __graft_entry__
        __graft_entry__.build()
    trackfit.load()
    return trackfit


def inputs(w, tb):
    h = W.paper_hits(tb, w)
    seed = S.seed_from_hits(h[..., :3], tb.n_hits, w.b_field)
    h[..., 12:15] = S.seed_features(seed, h[..., :3], tb.n_hits, w.b_field).astype(np.float32)
    return h


def run(T, model, blob, hits, n_hits, path=None, packed=False):
    dev = torch.device("cuda:0")
    B = len(n_hits)
    with T.Trackfit(model, blob) as tf:
        if path is not None:
            tf.set_path(path)
        out = torch.full((B, 5), -7.0, device=dev)
        q = torch.empty((B, 5, model.n_quantiles), device=dev)
        pooled = torch.empty((B, model.pooled_dim), device=dev)
        nh = torch.from_numpy(np.ascontiguousarray(n_hits)).to(dev)
        if packed:
            rows = np.concatenate([hits[b, :n_hits[b]] for b in range(B)])
            offs = np.concatenate([[0], np.cumsum(n_hits)]).astype(np.int64)
            tf.forward_packed(torch.from_numpy(rows).to(dev), torch.from_numpy(offs).to(dev), out)
        else:
            tf.forward(torch.from_numpy(np.ascontiguousarray(hits)).to(dev), nh, out, quantiles=q, pooled=pooled)
        torch.cuda.synchronize()
        st = tf.device_errors()
        used = tf.path
    return out.cpu().numpy(), q.cpu().numpy(), pooled.cpu().numpy(), st, used


# fp32 runs on the CUDA cores; fp16 on the packed-row tensor-core path by
# default and on the CUDA cores when asked (set_path 1)
@pytest.mark.parametrize("prec,force,want", [(W.PRECISION_FP32, None, "simt"), (W.PRECISION_FP16, None, "tcgen05-rows"),
                                             (W.PRECISION_FP16, 1, "simt")])
def test_transformer_matches_the_oracle(T, prec, force, want):
    w = W.workload("transformer", n_tracks=600, precision=prec)
    tb = W.gen_tracks(w)
    hits = inputs(w, tb)
    blob = W.gen_weights(w.model, w.weight_seed)
    got, q, pooled, st, path = run(T, w.model, blob, hits, tb.n_hits, path=force)
    assert st == (T.OK, 0)
    assert path.startswith(want), path
    cap = {}
    ref = O.forward(dataclasses.asdict(w.model), blob, hits, tb.n_hits, capture=cap)
    ok, msg = parity_ok(got, ref, prec)
    print(f"transformer {path} precision {prec}: {msg}")
    assert ok, msg
    ok, msg = parity_ok(q.reshape(len(got), -1), cap["quantiles"].reshape(len(got), -1), prec)
    assert ok, msg
    ok, msg = parity_ok(pooled, cap["pooled"], prec)
    assert ok, msg


@pytest.mark.parametrize("prec", [W.PRECISION_FP32, W.PRECISION_FP16])
def test_long_tracks_and_wide_heads(T, prec):
    """64 hits per track at d_model 128 (the attention CTA stages 64 x 257 floats,
    66 KB of shared memory), 2 heads of width 64, and a one-hit track; fp32 on the
    CUDA cores, fp16 on the packed-row tensor-core path (MLP width 256: one
    256-column tile; q, k, v: two tiles of 192)."""
    m = W.ModelConfig(max_hits=64, d_model=128, d_hidden=256, n_layers=2, topology=W.TOPOLOGY_ATTENTION,
                      n_heads=2, precision=prec)
    w = W.Workload("long", 120, m, layout="sweep", n_barrel=64, min_hits=64)
    tb = W.gen_tracks(w)
    n = tb.n_hits.copy()
    n[::7] = np.random.default_rng(3).integers(1, 64, len(n[::7]))
    n[5] = 1
    blob = W.gen_weights(m, 2)
    got, _, _, st, _ = run(T, m, blob, tb.hits, n)
    assert st == (T.OK, 0)
    ref = O.forward(dataclasses.asdict(m), blob, tb.hits, n)
    ok, msg = parity_ok(got, ref, prec)
    print(f"long tracks, precision {prec}: {msg}")
    assert ok, msg


def test_masking_order_and_packed_input_are_bit_exact(T):
    w = W.workload("transformer", n_tracks=300)
    tb = W.gen_tracks(w)
    hits = inputs(w, tb)
    blob = W.gen_weights(w.model, w.weight_seed)
    base = run(T, w.model, blob, hits, tb.n_hits)[0]
    nan = hits.copy()
    nan[np.arange(w.model.max_hits)[None, :] >= tb.n_hits[:, None]] = np.nan
    np.testing.assert_array_equal(run(T, w.model, blob, nan, tb.n_hits)[0], base)
    perm = np.random.default_rng(2).permutation(300)
    np.testing.assert_array_equal(run(T, w.model, blob, hits[perm], tb.n_hits[perm])[0], base[perm])
    np.testing.assert_array_equal(run(T, w.model, blob, hits, tb.n_hits, packed=True)[0], base)


def test_bad_counts_give_nan_rows(T):
    w = W.workload("transformer", n_tracks=40)
    tb = W.gen_tracks(w)
    hits = inputs(w, tb)
    n = tb.n_hits.copy()
    n[3], n[9] = 0, w.model.max_hits + 1
    blob = W.gen_weights(w.model, w.weight_seed)
    got, _, _, st, _ = run(T, w.model, blob, hits, n)
    assert st == (T.ERR_BAD_HITS, 2)
    assert np.all(np.isnan(got[[3, 9]]))
    good = np.setdiff1d(np.arange(40), [3, 9])
    ref = O.forward(dataclasses.asdict(w.model), blob, hits[good], n[good])
    ok, msg = parity_ok(got[good], ref, w.model.precision)
    assert ok, msg
