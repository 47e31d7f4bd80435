"""The paper's own model (Sec. 3.2: 15 features, d_model 128, two layers of width
192, concatenated directions, endpoint readout, fp16 operands) on the GPU against
the oracle, and the whole seed-guided forward (Sec. 3.1-3.3): the fp64 seed
writes its three residual features into the hit rows in place, the encoder reads
all 15, and the seed decode turns the heads' median corrections into track
parameters."""
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


def oracle_inputs(w, tb):
    """15-feature rows with the oracle's seed features (rounded to fp32) and the seed."""
    h = W.paper_hits(tb, w)
    seed = S.seed_from_hits(h[..., :3], tb.n_hits, w.b_field)
    h[..., 12:15] = S.seed_features(seed, h[..., :3], tb.n_hits, w.b_field).astype(np.float32)
    return h, seed


def gpu_encoder(T, model, blob, hits, n_hits, path=None):
    dev = torch.device("cuda:0")
    with T.Trackfit(model, blob) as tf:
        if path is not None:
            tf.set_path(path)
        B = len(n_hits)
        out = torch.full((B, 5), -7.0, device=dev)
        q = torch.empty((B, 5, model.n_quantiles), device=dev)
        tf.forward(torch.from_numpy(np.ascontiguousarray(hits)).to(dev), torch.from_numpy(n_hits).to(dev), out,
                   quantiles=q)
        torch.cuda.synchronize()
        st = tf.device_errors()
        path = tf.path
    assert st == (T.OK, 0)
    return out.cpu().numpy(), q.cpu().numpy(), path


# (operand precision, path): fp32 runs on the CUDA cores; fp16 on the packed-row
# tensor-core path by default and on the CUDA cores when asked (set_path 1)
@pytest.mark.parametrize("prec,path,want", [(W.PRECISION_FP32, None, "simt"), (W.PRECISION_FP16, None, "tcgen05-rows"),
                                            (W.PRECISION_FP16, 1, "simt")])
def test_paper_encoder_matches_the_oracle(T, prec, path, want):
    w = W.workload("paper", n_tracks=1000, precision=prec)
    tb = W.gen_tracks(w)
    hits, _ = oracle_inputs(w, tb)
    blob = W.gen_weights(w.model, w.weight_seed)
    got, q, used = gpu_encoder(T, w.model, blob, hits, tb.n_hits, path)
    assert used.startswith(want), used
    path = used
    cap = {}
    ref = O.forward(dataclasses.asdict(w.model), blob, hits, tb.n_hits, capture=cap)
    ok, msg = parity_ok(got, ref, prec)
    print(f"paper encoder {path}: {msg}")
    assert ok, msg
    ok, msg = parity_ok(q.reshape(len(got), -1), cap["quantiles"].reshape(len(got), -1), prec)
    assert ok, msg


@pytest.mark.parametrize("path", [None, 1])
def test_paper_encoder_masking_and_order(T, path):
    """NaN in the padded entries and a permuted batch change nothing, bit for bit,
    on the packed-row tensor-core path (every row's products are independent of
    the other rows, and each track's scan runs over its own rows in order) and on
    the CUDA cores."""
    w = W.workload("paper", n_tracks=300)
    tb = W.gen_tracks(w)
    hits, _ = oracle_inputs(w, tb)
    blob = W.gen_weights(w.model, w.weight_seed)
    base = gpu_encoder(T, w.model, blob, hits, tb.n_hits, path)[0]
    nan = hits.copy()
    nan[np.arange(w.model.max_hits)[None, :] >= tb.n_hits[:, None]] = np.nan
    np.testing.assert_array_equal(gpu_encoder(T, w.model, blob, nan, tb.n_hits, path)[0], base)
    perm = np.random.default_rng(2).permutation(300)
    got = gpu_encoder(T, w.model, blob, hits[perm], tb.n_hits[perm], path)[0]
    np.testing.assert_array_equal(got, base[perm])


def test_seed_guided_forward_matches_the_oracle(T):
    """Seed (fp64, features written into columns 12-14 in place) -> encoder (fp16
    operands) -> decode, all on the device, against the same chain in the oracle:
    the features where the foot point is unique, the heads' corrections at the
    fp16 bar, and the decoded parameters (seed + correction) to the corrections'
    error."""
    w = W.workload("paper", n_tracks=1000)
    tb = W.gen_tracks(w)
    hits_o, seed_o = oracle_inputs(w, tb)
    blob = W.gen_weights(w.model, w.weight_seed)
    dev = torch.device("cuda:0")
    hits = torch.from_numpy(W.paper_hits(tb, w)).to(dev)
    nh = torch.from_numpy(tb.n_hits).to(dev)
    seed = torch.empty((1000, 5), dtype=torch.float64, device=dev)
    T.seed(hits, nh, w.b_field, seed, in_place_at=12)
    with T.Trackfit(w.model, blob) as tf:
        corr = torch.empty((1000, 5), device=dev)
        tf.forward(hits, nh, corr)
        out = torch.empty((1000, 5), device=dev)
        T.decode(seed, corr, out)
        torch.cuda.synchronize()
    h, sd, c, o = hits.cpu().numpy(), seed.cpu().numpy(), corr.cpu().numpy(), out.cpu().numpy()
    np.testing.assert_array_equal(np.isnan(sd), np.isnan(seed_o))
    np.testing.assert_array_equal(h[..., :12], hits_o[..., :12])   # the seed wrote only its own columns
    valid = np.arange(w.model.max_hits)[None, :] < tb.n_hits[:, None]
    near = valid & (np.abs(np.sinh(hits_o[..., 12])) < 50.0) & (np.abs(np.sinh(hits_o[..., 13])) < 50.0)
    assert np.max(np.abs(h[..., 12:14][near] - hits_o[..., 12:14][near])) < 2e-6
    corr_o = O.forward(dataclasses.asdict(w.model), blob, hits_o, tb.n_hits)
    ok_seed = ~np.isnan(seed_o[:, 0])
    ok, msg = parity_ok(c[ok_seed], corr_o[ok_seed], w.model.precision)
    print(f"seed-guided forward, corrections: {msg}")
    assert ok, msg
    dec_o = S.decode(seed_o, corr_o)
    d = np.abs(o[ok_seed] - dec_o[ok_seed])
    d[:, 2] = np.minimum(d[:, 2], 2 * np.pi - d[:, 2])
    # q/p = q/p_seed + r (|q/p_seed| + 0.02): its correction enters scaled
    gain = np.ones_like(d)
    gain[:, 4] = np.abs(seed_o[ok_seed, 4]) + 0.02
    scale = np.abs(c[ok_seed] - corr_o[ok_seed]) * gain + 1e-6 * np.maximum(np.abs(dec_o[ok_seed]), 1.0)
    assert np.all(d <= scale), np.max(d - scale, axis=0)
    assert np.all(np.isnan(o[~ok_seed]))


@pytest.mark.parametrize("T_,L,pool,n_tracks", [(64, 3, W.POOL_ENDPOINTS, 700), (24, 2, W.POOL_MEAN, 500),
                                                (8, 1, W.POOL_ENDPOINTS, 600)])
def test_concatenation_shapes_on_the_tensor_cores(T, T_, L, pool, n_tracks):
    """The concatenation topology with fp16 operands on the packed-row tensor-core
    path beyond the paper's shape: tracks of 1-64 hits (a track's rows cross
    128-row tiles), three layers, mean pooling, invalid counts; against the oracle
    at the fp16 bar, invalid tracks NaN."""
    m = W.ModelConfig(max_hits=T_, d_model=128, d_hidden=192, n_layers=L, precision=W.PRECISION_FP16, pool=pool,
                      topology=W.TOPOLOGY_CONCAT)
    w = W.Workload("c", n_tracks, m, layout="sweep", n_barrel=T_, min_hits=T_)
    tb = W.gen_tracks(w)
    n = np.random.default_rng(T_ + L).integers(1, T_ + 1, n_tracks).astype(np.int32)
    n[:40] = T_
    n[40:60] = 1
    n[77], n[300] = 0, T_ + 1
    blob = W.gen_weights(m, 5)
    dev = torch.device("cuda:0")
    with T.Trackfit(m, blob) as tf:
        out = torch.full((n_tracks, 5), -7.0, device=dev)
        tf.forward(torch.from_numpy(tb.hits).to(dev), torch.from_numpy(n).to(dev), out)
        torch.cuda.synchronize()
        st = tf.device_errors()
        path = tf.path
    got = out.cpu().numpy()
    assert path.startswith("tcgen05-rows"), path
    assert st == (T.ERR_BAD_HITS, 2)
    assert np.all(np.isnan(got[[77, 300]]))
    good = np.setdiff1d(np.arange(n_tracks), [77, 300])
    ref = O.forward(dataclasses.asdict(m), blob, tb.hits[good], n[good])
    ok, msg = parity_ok(got[good], ref, W.PRECISION_FP16)
    print(f"concatenation T={T_} L={L} pool={pool}: {msg}")
    assert ok, msg
