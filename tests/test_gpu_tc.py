"""tcgen05 path unit checks: the UMMA operand layouts (TMA-staged K-major
weights x thread-written MN-major activations -> TMEM) against a plain fp32
matrix product of the same bf16 values."""
import numpy as np
import pytest

from paper_2609_32479_gb300 import workloads as W

pytestmark = pytest.mark.gpu
torch = pytest.importorskip("torch")


@pytest.fixture(scope="module")
def tf():
    from paper_2609_32479_gb300 import trackfit
    m = W.workload("medium").model
    h = trackfit.Trackfit(m, W.gen_weights(m, 1))
    yield h
    h.close()


@pytest.mark.parametrize("K", [64, 128, 192, 256])
def test_umma_probe_matches_matmul(tf, K):
    from paper_2609_32479_gb300 import trackfit
    g = torch.Generator().manual_seed(K)
    A = torch.randn(128, K, generator=g).to(torch.bfloat16)
    B = torch.randn(K, 128, generator=g).to(torch.bfloat16)
    # structured rows/columns make a layout slip visible even where random data averages out
    A[5, :] = 0
    A[5, 3] = 1
    B[:, 77] = torch.arange(K, dtype=torch.float32).to(torch.bfloat16)
    dev = torch.device("cuda:0")
    Ad = A.view(torch.int16).contiguous().to(dev)
    Bd = B.view(torch.int16).contiguous().to(dev)
    D = torch.full((128, 128), float("nan"), device=dev)
    trackfit.debug_umma(tf, Ad, Bd, D)
    torch.cuda.synchronize()
    ref = (A.float() @ B.float()).numpy()
    got = D.cpu().numpy()
    np.testing.assert_allclose(got[5], B.float().numpy()[3], rtol=0, atol=0)
    np.testing.assert_allclose(got, ref, rtol=1e-5, atol=1e-4 * np.sqrt(K))
