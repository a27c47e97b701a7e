"""Every output of whole 36-layer decode-step weight passes (q|k|v and gate|up fused: 144 GEMVs)
against the oracle, in the forms the bench times: the CUDA graph of laq_gemm_wxg128 launches and
the planned pass (laq_pass_run).

The other full-size tests sample a few tiles of a few layers; here the oracle quantizes every
projection's fp16 weights (regenerated from their seeds) and multiplies every output, with its
routines split over the host's cores (bit-identical to the single-threaded definitions, pinned
in tests/test_oracle_pins.py).  Scales and zeros must match bit for bit, every Y within the
stated tolerance.  Cases: the Qwen3-4B W3 M = 1 pass in both forms, W4, the batch paths at
M = 4, 8 (W4: the down projection in 4-warp CTAs with a cluster of 8) and 16 (two MMAs per k16
step), a planned W4 M = 2 pass, and the Qwen3-8B pass with 1 % outlier weights in both forms
(the graph's gate|up in three waves of 2-tile CTAs, its down unclustered).
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


CASES = [
    ("qwen3-4b", 3, 1, False),
    ("qwen3-4b", 3, 1, True),
    ("qwen3-4b", 4, 1, False),
    ("qwen3-4b", 3, 4, False),
    ("qwen3-4b", 3, 16, False),
    ("qwen3-4b", 4, 2, True),
    ("qwen3-4b", 4, 8, False),
    ("qwen3-8b", 3, 1, True),
    ("qwen3-8b", 3, 1, False),
]


@pytest.mark.parametrize("model,bits,M,planned", CASES,
                         ids=[f"{m}-w{b}-m{M}-{'planned' if p else 'graph'}"
                              for m, b, M, p in CASES])
def test_whole_pass_every_output(model, bits, M, planned):
    wp = WeightPass(model=model, bits=bits, M=M, fuse=True, planned=planned,
                    outliers=model == "qwen3-8b")
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
        codes, s, z = co.quantize_rtn_threads(W, bits)
        assert np.array_equal(q.s.cpu().numpy().view(np.uint16), s.view(np.uint16)), (layer, name)
        assert np.array_equal(q.z.cpu().numpy(), z), (layer, name)
        yref = co.gemm_threads(wp.X[idx].cpu().numpy(), codes, s, z)
        y = Yall[yo:yo + M * q.N].reshape(M, q.N)
        yo += M * q.N
        err = np.abs(y - yref).max()
        assert err <= tolerance(yref), (layer, name, err, tolerance(yref))
        worst = max(worst, err / tolerance(yref))
    assert yo == Yall.size
    print(f"worst |Y - Y_ref| / tolerance over the pass: {worst:.3f}")
