"""laq_gemm_chain_static: the chain for callers that cannot allocate device memory.

Such callers (a host framework that owns every device allocation and hands a plug-in no
scratch, or a decode loop that may not call cudaMalloc once it runs) get the chain with the
library's own static scratch.  This test calls it through the C ABI twice in a row and compares
each result with laq_gemm_chain's on the same entries, within the GEMV tolerance of the other
tests.  It sits in its own file, collected last, and needs nothing from earlier tests.
"""
import numpy as np
import pytest
import torch

import paper_2605_08755_gb300 as laq
from paper_2605_08755_gb300 import inputs
from tests.conftest import tolerance

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def built():
    import __graft_entry__
    __graft_entry__.build()


def quantized(K, N, bits, seed):
    W = torch.from_numpy(inputs.weights(K, N, seed)).cuda()
    codes, s, z = laq.laq_quantize_rtn(W, bits)
    return laq.laq_pack(codes, bits), s, z


@pytest.mark.parametrize("bits,M", [(3, 1), (4, 2)])
def test_static_scratch_chain_matches_workspace_chain(bits, M):
    # three stages with real dependencies: x -> (a, b) -> c(a)
    dims = [(2560, 4096), (2560, 1024), (4096, 2560)]
    lins = [quantized(K, N, bits, 50 + i) for i, (K, N) in enumerate(dims)]
    X = torch.from_numpy(inputs.activations(M, 2560, seed=3)).cuda()
    Ya = torch.empty((M, 4096), dtype=torch.float16, device="cuda")
    Yb = torch.empty((M, 1024), dtype=torch.float16, device="cuda")
    Yc = torch.empty((M, 2560), dtype=torch.float16, device="cuda")
    spec = laq.Chain([(X, *lins[0], bits, Ya, 1), (X, *lins[1], bits, Yb, 0),
                      (Ya, *lins[2], bits, Yc, 1)])
    ws = laq.chain_workspace(3, "cuda")
    spec.run(ws)
    ref = [Y.clone() for Y in (Ya, Yb, Yc)]
    assert laq.chain_status(ws) == 0
    for call in range(2):
        for Y in (Ya, Yb, Yc):
            Y.fill_(float("nan"))
        spec.run_static()
        torch.cuda.synchronize()
        for Y, R in zip((Ya, Yb, Yc), ref):
            r = R.cpu().numpy().astype(np.float64)
            y = Y.cpu().numpy().astype(np.float64)
            assert np.isfinite(y).all(), call
            assert np.abs(y - r).max() <= tolerance(r), call
