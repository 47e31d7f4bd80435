"""Failure detection without a GPU fault.

1. A bounded wait inside the fused tensor-core kernel that runs out: a test hook
   lowers the wait limit and makes the first CTA's loader warp hold back one
   metadata hand-over past it.  The kernel must record the timeout, drain and
   return (no hang), trackfit_device_errors must report TRACKFIT_ERR_TIMEOUT, and
   the handle and the device must stay usable: later forwards are bit-identical
   to those of a fresh handle.
2. A device allocation that fails inside trackfit_create (or the staging buffers
   of trackfit_forward_host): the call returns TRACKFIT_ERR_OOM and frees what it
   had allocated, for every allocation in turn.
"""
import gc
import time

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


def _inputs(name, n):
    w = W.workload(name, n_tracks=n)
    tb = W.gen_tracks(w)
    dev = torch.device("cuda:0")
    return w, W.gen_weights(w.model, w.weight_seed), torch.from_numpy(tb.hits).to(dev), \
        torch.from_numpy(tb.n_hits).to(dev)


@pytest.mark.parametrize("name,n", [("medium", 3000), ("large", 2000)])
def test_expired_wait_reports_timeout_and_the_handle_recovers(T, name, n):
    w, blob, hits, nh = _inputs(name, n)
    with T.Trackfit(w.model, blob) as fresh:
        ref = torch.empty((n, 5), device=hits.device)
        fresh.forward(hits, nh, ref)
        torch.cuda.synchronize()
        assert fresh.device_errors() == (T.OK, 0)
        ref = ref.cpu().numpy()
    with T.Trackfit(w.model, blob) as tf:
        assert tf.path.startswith("tcgen05")
        tf.debug_wait_limit(50_000_000, hold_tile=0)          # 50 ms, CTA 0 holds its first tile
        out = torch.full((n, 5), -7.0, device=hits.device)
        t0 = time.perf_counter()
        tf.forward(hits, nh, out)
        torch.cuda.synchronize()
        took = time.perf_counter() - t0
        st, nbad = tf.device_errors()
        assert st == T.ERR_TIMEOUT, st
        assert took < 5.0, f"the aborted forward took {took:.1f} s"
        # the counters were reset and the device is fine: the same handle with the
        # normal limit reproduces the fresh handle's result bit for bit
        tf.debug_wait_limit(0, hold_tile=-1)
        for _ in range(2):
            out = torch.full((n, 5), -7.0, device=hits.device)
            tf.forward(hits, nh, out)
            torch.cuda.synchronize()
            assert tf.device_errors() == (T.OK, 0)
            np.testing.assert_array_equal(out.cpu().numpy(), ref)


def test_wait_limit_hook_is_rejected_on_the_cuda_core_path(T):
    w, blob, _, _ = _inputs("tiny", 8)
    with T.Trackfit(w.model, blob) as tf:
        with pytest.raises(T.TrackfitError) as ei:
            tf.debug_wait_limit(1_000_000, 0)
        assert ei.value.status == T.ERR_UNSUPPORTED
    w, blob, _, _ = _inputs("medium", 8)
    with T.Trackfit(w.model, blob) as tf:
        for bad in ((-1, -1), (0, -2)):
            with pytest.raises(T.TrackfitError) as ei:
                tf.debug_wait_limit(*bad)
            assert ei.value.status == T.ERR_INVALID_ARG


@pytest.mark.parametrize("name", ["small", "medium"])
def test_failed_allocation_in_create_returns_oom_and_frees_everything(T, name):
    w, blob, hits, nh = _inputs(name, 64)
    gc.collect()
    torch.cuda.synchronize()
    live0, _ = T.debug_alloc(0)
    with T.Trackfit(w.model, blob) as tf:
        live1, n_alloc = T.debug_alloc(0)
        assert live1 - live0 == n_alloc >= 3
        out = torch.empty((64, 5), device=hits.device)
        tf.forward(hits, nh, out)
        torch.cuda.synchronize()
        ref = out.cpu().numpy()
    assert T.debug_alloc(0)[0] == live0
    for k in range(1, n_alloc + 1):
        T.debug_alloc(k)
        with pytest.raises(T.TrackfitError) as ei:
            T.Trackfit(w.model, blob)
        assert ei.value.status == T.ERR_OOM, (k, ei.value.status)
        live, att = T.debug_alloc(0)
        assert att == k, (k, att)                 # it stopped at the failed allocation
        assert live == live0, f"allocation {k} failed: {live - live0} allocations leaked"
    # nothing armed any more: a handle works as before
    with T.Trackfit(w.model, blob) as tf:
        out = torch.empty((64, 5), device=hits.device)
        tf.forward(hits, nh, out)
        torch.cuda.synchronize()
        np.testing.assert_array_equal(out.cpu().numpy(), ref)
    assert T.debug_alloc(0)[0] == live0


def test_failed_staging_allocation_in_forward_host_returns_oom(T):
    w = W.workload("medium", n_tracks=500)
    tb = W.gen_tracks(w)
    blob = W.gen_weights(w.model, w.weight_seed)
    with T.Trackfit(w.model, blob) as tf:
        live0, _ = T.debug_alloc(0)
        out = np.zeros((500, 5), np.float32)
        for k in (1, 2, 3):
            T.debug_alloc(k)
            with pytest.raises(T.TrackfitError) as ei:
                tf.forward_host(tb.hits, tb.n_hits, out)
            assert ei.value.status == T.ERR_OOM
            assert T.debug_alloc(0)[0] == live0
        tf.forward_host(tb.hits, tb.n_hits, out)     # and then it works
        assert np.all(np.isfinite(out))
        assert T.debug_alloc(0)[0] == live0 + 3
