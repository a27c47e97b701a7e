"""The benchmark workloads at full size, in the launch configuration bench.py times (the
library's own plan, one CUDA graph per pass), checked against the CPU oracle.

Workloads (synthetic stand-ins for Qwen3 weights: W ~ N(0, 0.02^2), X ~ N(0, 1)):
  1. one 1024 x 1024 W3G128 linear, M = 1 (fully checked);
  2. one Qwen3-4B-shaped decoder layer (q, k, v, o, gate, up, down), W3, M = 1 (fully checked);
  3. the 36-layer Qwen3-4B-shaped pass, W3, M = 1, one CUDA graph (sampled);
  4. the same pass at W3 and W4 for M in {1, 2, 4, 8, 16} (sampled);
  5. the 36-layer Qwen3-8B-shaped pass with 1% x20 outliers, W3, M in {1, 16} (sampled).
Sampled checks regenerate the fp16 weights of chosen projections from their seeds and compare
whole 16-column tiles: s, z and packed records bit-exact, Y within the stated tolerance.
"""
import numpy as np
import pytest
import torch

from oracle import c_oracle as co
from paper_2605_08755_gb300 import inputs
from paper_2605_08755_gb300.weight_pass import WeightPass, shapes
from tests.conftest import tolerance

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def built():
    import __graft_entry__
    __graft_entry__.build()


def check_projection(wp, idx, tiles=None):
    layer, members, name, q = wp.linears[idx]
    K, N, bits = q.K, q.N, q.bits
    T, G = N // 16, K // 128
    rec = 256 * bits           # bytes of one 16-column x 128-row record
    if tiles is None:
        tiles = list(range(T))
    W = wp.weight(layer, members).cpu().numpy()
    X = wp.X[idx].cpu().numpy()
    Y = wp.Y[idx].cpu().numpy().astype(np.float64)
    s_gpu = q.s.cpu().numpy().view(np.uint16)
    z_gpu = q.z.cpu().numpy()
    packed = q.packed.cpu().numpy()
    cols = np.concatenate([np.arange(16 * t, 16 * t + 16) for t in tiles])
    codes, s, z = co.quantize_rtn(np.ascontiguousarray(W[:, cols]), bits)
    assert np.array_equal(s_gpu[:, cols], s.view(np.uint16)), (layer, name)
    assert np.array_equal(z_gpu[:, cols], z), (layer, name)
    for i, t in enumerate(tiles):
        sub = np.ascontiguousarray(codes[:, 16 * i:16 * i + 16])
        ref = co.pack(sub, bits).view(np.uint8)
        got = packed[t * G * rec:(t + 1) * G * rec]
        assert np.array_equal(got, ref), (layer, name, t)
    yref = co.gemm(X, codes, s, z)
    err = np.abs(Y[:, cols] - yref).max()
    assert err <= tolerance(yref), (layer, name, err, tolerance(yref))


def replay(wp):
    g = wp.capture()
    wp.Ybuf.zero_()
    g.replay()
    torch.cuda.synchronize()
    return g


def test_single_linear_1024():
    wp = WeightPass(model="qwen3-4b", bits=3, M=1, layers=1)
    # replace the pass by the single 1024 x 1024 linear of the first workload
    from paper_2605_08755_gb300 import laq_gemm_wxg128
    from paper_2605_08755_gb300.weight_pass import QuantLinear
    W = inputs.weights(1024, 1024, seed=0)
    X = inputs.activations(1, 1024, seed=0)
    ql = QuantLinear(torch.from_numpy(W).cuda(), 3)
    Y = laq_gemm_wxg128(torch.from_numpy(X).cuda(), ql.packed, ql.s, ql.z, 3)
    torch.cuda.synchronize()
    codes, s, z = co.quantize_rtn(W, 3)
    assert np.array_equal(ql.s.cpu().numpy().view(np.uint16), s.view(np.uint16))
    assert np.array_equal(ql.z.cpu().numpy(), z)
    assert np.array_equal(ql.packed.cpu().numpy(), co.pack(codes, 3).view(np.uint8))
    yref = co.gemm(X, codes, s, z)
    assert np.abs(Y.cpu().numpy().astype(np.float64) - yref).max() <= tolerance(yref)
    del wp


def test_one_qwen3_4b_layer_fully():
    wp = WeightPass(model="qwen3-4b", bits=3, M=1, layers=1)
    replay(wp)
    for idx in range(wp.launches):
        check_projection(wp, idx)


def _sampled(wp, layers):
    for idx, (layer, members, name, q) in enumerate(wp.linears):
        if layer in layers:
            T = q.N // 16
            check_projection(wp, idx, tiles=sorted({0, T // 2, T - 1}))


def test_qwen3_4b_pass_w3_m1():
    wp = WeightPass(model="qwen3-4b", bits=3, M=1)
    assert wp.launches == 252
    replay(wp)
    _sampled(wp, layers={0, 17, 35})


@pytest.mark.parametrize("bits", [3, 4])
@pytest.mark.parametrize("M", [1, 2, 4, 8, 16])
def test_qwen3_4b_pass_batch_sweep(bits, M):
    wp = WeightPass(model="qwen3-4b", bits=bits, M=M)
    replay(wp)
    _sampled(wp, layers={5, 30})


@pytest.mark.parametrize("bits,M", [(3, 1), (4, 1), (3, 8), (3, 16)])
def test_qwen3_4b_fused_pass(bits, M):
    """q|k|v and gate|up as single GEMVs over concatenated columns (4 launches per layer)."""
    wp = WeightPass(model="qwen3-4b", bits=bits, M=M, fuse=True)
    assert wp.launches == 4 * 36
    assert [n for _, _, n, _ in wp.linears[:4]] == ["qkv", "o", "gate_up", "down"]
    replay(wp)
    _sampled(wp, layers={0, 35})


@pytest.mark.parametrize("M", [1, 16])
def test_qwen3_8b_pass_with_outliers(M):
    wp = WeightPass(model="qwen3-8b", bits=3, M=M, outliers=True)
    assert [(n, K, N) for n, K, N in shapes("qwen3-8b")][6] == ("down", 12288, 4096)
    replay(wp)
    _sampled(wp, layers={0, 35})
