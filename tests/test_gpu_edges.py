"""Edge cases of the tensor-core path against the oracle: tracks of every length
from 1 to max_hits (a one-hit track is its own first and last column, and the
reverse scan restarts there; short tracks fill a slab to its 16-track limit
before its 64 columns), a batch of one track, and a batch one track longer
than the internal pooled-buffer chunk of 1,048,576 tracks.  Masks, packing and
chunking must not change any result: those checks are bit-exact."""
import dataclasses

import numpy as np
import pytest

from oracle import fp32_emulation as E
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


def run(T, model, blob, hits, n_hits):
    dev = torch.device("cuda:0")
    with T.Trackfit(model, blob) as tf:
        h = torch.from_numpy(np.ascontiguousarray(hits)).to(dev)
        n = torch.from_numpy(np.ascontiguousarray(n_hits)).to(dev)
        out = torch.full((n.shape[0], 5), -7.0, dtype=torch.float32, device=dev)
        tf.forward(h, n, out)
        torch.cuda.synchronize()
        st, nbad = tf.device_errors()
        path = tf.path
    assert st == 0 and nbad == 0
    return out.cpu().numpy(), path


def references(model, blob, hits, n_hits):
    """The oracle's outputs and the fp32 emulation's (every accumulation order)."""
    cfg = dataclasses.asdict(model)
    return O.forward(cfg, blob, hits, n_hits), [E.forward(cfg, blob, hits, n_hits, order=o) for o in E.ORDERS]


def ragged(name, n, seed):
    """Generated tracks of the workload with hit counts redrawn uniformly in
    [1, max_hits]; hits past a track's generated ones are zero rows (still valid
    hits for both sides)."""
    w = W.workload(name, n_tracks=n)
    tb = W.gen_tracks(w)
    n_hits = np.random.default_rng(seed).integers(1, w.model.max_hits + 1, n).astype(np.int32)
    return w, tb.hits, n_hits


@pytest.mark.parametrize("name,n", [("medium", 900), ("large", 400)])
def test_every_track_length_from_one_to_max_hits(T, name, n):
    w, hits, n_hits = ragged(name, n, seed=21)
    assert set(np.unique(n_hits)) == set(range(1, w.model.max_hits + 1))
    blob = W.gen_weights(w.model, w.weight_seed)
    got, path = run(T, w.model, blob, hits, n_hits)
    assert path.startswith("tcgen05")
    ref, em = references(w.model, blob, hits, n_hits)
    ok, msg = parity_ok(got, ref, w.model.precision, emul=em)
    print(f"{name} n_b in [1, {w.model.max_hits}]: {msg}")
    assert np.all(np.isfinite(got))
    assert ok, msg
    # the same tracks permuted, and split over three calls: bit-identical
    perm = np.random.default_rng(5).permutation(n)
    np.testing.assert_array_equal(run(T, w.model, blob, hits[perm], n_hits[perm])[0], got[perm])
    parts = [run(T, w.model, blob, hits[a:b], n_hits[a:b])[0] for a, b in ((0, 1), (1, n // 2), (n // 2, n))]
    np.testing.assert_array_equal(np.concatenate(parts), got)


def test_slabs_of_sixteen_one_hit_tracks(T):
    """Only one-hit tracks: every slab holds its maximum of 16 tracks in 16 of its
    64 columns, every column is both a first and a last hit."""
    w = W.workload("medium", n_tracks=500)
    tb = W.gen_tracks(w)
    n_hits = np.ones(500, np.int32)
    blob = W.gen_weights(w.model, w.weight_seed)
    got, _ = run(T, w.model, blob, tb.hits, n_hits)
    ref, em = references(w.model, blob, tb.hits, n_hits)
    ok, msg = parity_ok(got, ref, w.model.precision, emul=em)
    assert ok, msg


@pytest.mark.parametrize("name", ["medium", "large"])
def test_single_track_batch(T, name):
    w = W.workload(name, n_tracks=40)
    tb = W.gen_tracks(w)
    blob = W.gen_weights(w.model, w.weight_seed)
    batch, _ = run(T, w.model, blob, tb.hits, tb.n_hits)
    for b in (0, 17, 39):
        one, _ = run(T, w.model, blob, tb.hits[b:b + 1], tb.n_hits[b:b + 1])
        np.testing.assert_array_equal(one[0], batch[b])


def test_batch_crossing_the_pooled_buffer_chunk(T):
    """1,048,577 tracks: the library runs two launches (1,048,576 + 1 tracks)
    through its internal pooled buffer; outputs equal those of the two halves run
    on their own, and sampled tracks on both sides of the boundary match the
    oracle."""
    B = 1048577
    w = W.workload("large", n_tracks=B)
    tb = W.gen_tracks(w)
    blob = W.gen_weights(w.model, w.weight_seed)
    got, _ = run(T, w.model, blob, tb.hits, tb.n_hits)
    tail, _ = run(T, w.model, blob, tb.hits[B - 3:], tb.n_hits[B - 3:])
    np.testing.assert_array_equal(got[B - 3:], tail)
    head, _ = run(T, w.model, blob, tb.hits[:5000], tb.n_hits[:5000])
    np.testing.assert_array_equal(got[:5000], head)
    idx = np.array(sorted(set(range(B - 200, B)) | set(range(0, 100))))
    ref, em = references(w.model, blob, tb.hits[idx], tb.n_hits[idx])
    ok, msg = parity_ok(got[idx], ref, w.model.precision, emul=em)
    assert ok, msg
