"""The packed, unpadded input (Sec. 3.5) through trackfit_forward_packed: the
same tracks give bit-identical results to the padded entry point on both kernel
paths, whatever the rows before the first track; tracks whose row range is
empty, too long or outside the hit array get NaN rows and are counted."""
import numpy as np
import pytest

from paper_2609_32479_gb300 import workloads as W

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


def pack(hits, n_hits, lead=0):
    """Packed rows (with `lead` junk rows first) and offsets [B + 1]."""
    rows = [np.full((lead, 5), 123.0, np.float32)] + [hits[b, :n_hits[b]] for b in range(len(n_hits))]
    offs = np.concatenate([[lead], lead + np.cumsum(n_hits)]).astype(np.int64)
    return np.ascontiguousarray(np.concatenate(rows)), offs


def run_both(T, w, blob, tb, path, lead):
    dev = torch.device("cuda:0")
    with T.Trackfit(w.model, blob) as tf:
        if path:
            tf.set_path(path)
        B = len(tb.n_hits)
        a = torch.full((B, 5), -7.0, device=dev)
        tf.forward(torch.from_numpy(tb.hits).to(dev), torch.from_numpy(tb.n_hits).to(dev), a)
        ph, po = pack(tb.hits, tb.n_hits, lead)
        b = torch.full((B, 5), -7.0, device=dev)
        tf.forward_packed(torch.from_numpy(ph).to(dev), torch.from_numpy(po).to(dev), b)
        torch.cuda.synchronize()
        st = tf.device_errors()
        return a.cpu().numpy(), b.cpu().numpy(), st, tf.path


@pytest.mark.parametrize("name,n,path", [("tiny", 256, 0), ("small", 3000, 0), ("medium", 3000, 0),
                                         ("large", 2000, 0), ("sweep64", 500, 0), ("medium", 700, 1)])
def test_packed_matches_padded_bit_exactly(T, name, n, path):
    w = W.workload(name, n_tracks=n)
    tb = W.gen_tracks(w)
    blob = W.gen_weights(w.model, w.weight_seed)
    for lead in (0, 37):
        padded, packed, st, p = run_both(T, w, blob, tb, path, lead)
        assert st == (T.OK, 0)
        np.testing.assert_array_equal(packed, padded)
    assert p.startswith("simt" if path == 1 or w.model.precision == 0 else "tcgen05")


@pytest.mark.parametrize("name", ["small", "medium"])
def test_packed_invalid_ranges(T, name):
    w = W.workload(name, n_tracks=40)
    tb = W.gen_tracks(w)
    blob = W.gen_weights(w.model, w.weight_seed)
    dev = torch.device("cuda:0")
    ph, po = pack(tb.hits, tb.n_hits)
    with T.Trackfit(w.model, blob) as tf:
        ref = torch.empty((40, 5), device=dev)
        tf.forward_packed(torch.from_numpy(ph).to(dev), torch.from_numpy(po).to(dev), ref)
        ref = ref.cpu().numpy()
        bad = po.copy()
        bad[5] = bad[4]                       # track 4 empty (track 5 starts where 4 began)
        bad[11] = bad[10] + w.model.max_hits + 1   # track 10 too long
        bad[20] = -3                          # track 19 ends before it starts, 20 starts before row 0
        out = torch.empty((40, 5), device=dev)
        n_rows = ph.shape[0]
        tf.forward_packed(torch.from_numpy(ph).to(dev), torch.from_numpy(bad).to(dev), out)
        torch.cuda.synchronize()
        st, nbad = tf.device_errors()
        got = out.cpu().numpy()
        d = bad[1:] - bad[:-1]
        invalid = (d < 1) | (d > w.model.max_hits) | (bad[:-1] < 0) | (bad[1:] > n_rows)
        assert nbad == int(invalid.sum()) and st == T.ERR_BAD_HITS
        assert np.all(np.isnan(got[invalid]))
        same = ~invalid & (d == tb.n_hits) & (bad[:-1] == po[:-1])
        np.testing.assert_array_equal(got[same], ref[same])
        # a range past the end of the hit array is invalid too
        short = torch.from_numpy(ph[:-1].copy()).to(dev)
        tf.forward_packed(short, torch.from_numpy(po).to(dev), out)
        torch.cuda.synchronize()
        st, nbad = tf.device_errors()
        assert nbad == 1 and np.all(np.isnan(out.cpu().numpy()[-1]))
