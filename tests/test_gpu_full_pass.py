"""Every output of the 36-layer Qwen3-4B-shaped pass (W3G128, M = 1, q|k|v and gate|up fused:
144 GEMVs) against the oracle, in both forms the bench times: the CUDA graph of
laq_gemm_wxg128 launches and the planned pass (laq_pass_run).

The other full-size tests sample a few tiles of a few layers; here the oracle quantizes every
projection's fp16 weights (regenerated from their seeds) and multiplies every output, with its
routines split over the host's cores (bit-identical to the single-threaded definitions, pinned
in tests/test_oracle_pins.py).  Scales and zeros must match bit for bit, every Y within the
stated tolerance.
"""
import numpy as np
import pytest
import torch

from oracle import c_oracle as co
from paper_2605_08755_gb300.weight_pass import WeightPass
from tests.conftest import tolerance

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def built():
    import __graft_entry__
    __graft_entry__.build()


@pytest.mark.parametrize("planned", [False, True], ids=["graph_fused", "planned_fused"])
def test_qwen3_4b_pass_every_output(planned):
    wp = WeightPass(model="qwen3-4b", bits=3, M=1, fuse=True, planned=planned)
    assert wp.launches == (1 if planned else 144)
    g = wp.capture()
    wp.Ybuf.fill_(float("nan"))
    g.replay()
    torch.cuda.synchronize()
    if planned:
        assert wp.plan.status() == 0
    Yall = wp.Ybuf.cpu().numpy().astype(np.float64)
    yo = 0
    worst = 0.0
    for idx, (layer, members, name, q) in enumerate(wp.linears):
        W = wp.weight(layer, members).cpu().numpy()
        codes, s, z = co.quantize_rtn_threads(W, 3)
        assert np.array_equal(q.s.cpu().numpy().view(np.uint16), s.view(np.uint16)), (layer, name)
        assert np.array_equal(q.z.cpu().numpy(), z), (layer, name)
        yref = co.gemm_threads(wp.X[idx].cpu().numpy(), codes, s, z)
        y = Yall[yo:yo + q.N].reshape(1, q.N)
        yo += q.N
        err = np.abs(y - yref).max()
        assert err <= tolerance(yref), (layer, name, err, tolerance(yref))
        worst = max(worst, err / tolerance(yref))
    assert yo == Yall.size
    print(f"worst |Y - Y_ref| / tolerance over the pass: {worst:.3f}")
