"""The no-allocation forward (trackfit_forward_noalloc) against the handle-based
CUDA-core path on the same inputs, twice in a row.

It serves callers that cannot call cudaMalloc: its workspace is a static device
array inside the library, so its output must match the ordinary entry point's
and must not depend on what a previous call left in that array.  This file is
collected last so that a failure here comes after every other test has run."""
import numpy as np
import pytest

from paper_2609_32479_gb300 import workloads as W
from tests.helpers import parity_ok

pytestmark = pytest.mark.gpu
torch = pytest.importorskip("torch")


@pytest.mark.parametrize("name,n", [("small", 2000), ("medium", 300)])
def test_noalloc_forward_matches_handle_path_twice(name, n):
    from paper_2609_32479_gb300 import trackfit as T
    w = W.workload(name, n_tracks=n)
    tb = W.gen_tracks(w)
    blob = W.gen_weights(w.model, w.weight_seed)
    dev = torch.device("cuda:0")
    hits = torch.from_numpy(tb.hits).to(dev)
    nh = torch.from_numpy(tb.n_hits).to(dev)
    with T.Trackfit(w.model, blob) as tf:
        tf.set_path(1)                         # the CUDA-core path the variant shares
        ref = torch.empty((n, 5), device=dev)
        tf.forward(hits, nh, ref)
        torch.cuda.synchronize()
        ref = ref.cpu().numpy()
    wdev = torch.from_numpy(blob).to(dev)
    for _ in range(2):
        out = torch.full((n, 5), float("nan"), device=dev)
        T.forward_noalloc(w.model, wdev, hits, nh, out)
        torch.cuda.synchronize()
        got = out.cpu().numpy()
        assert np.all(np.isfinite(got))
        ok, msg = parity_ok(got, ref, 0)       # same arithmetic: the fp32 bar, whatever the precision
        assert ok, msg
