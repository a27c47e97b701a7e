"""laq_gemm_chain (one persistent launch for a list of GEMVs) against the oracle.

Every entry's Y must satisfy the GEMV tolerance against the oracle's fp64 product of the
oracle's own codes, scales and zeros (tests.conftest.tolerance).  The dependency tests feed one
entry's Y to the next entry as X, with every Y pre-filled with NaN, so an entry that read its
input before its producer finished would propagate NaN; the oracle recomputes the chain from
its own fp16-rounded intermediates.
"""
import numpy as np
import pytest
import torch

import paper_2605_08755_gb300 as laq
from oracle import c_oracle as co
from paper_2605_08755_gb300 import inputs
from paper_2605_08755_gb300.weight_pass import WeightPass
from tests.conftest import tolerance
from tests.test_gpu_workloads import _sampled, check_projection

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def built():
    import __graft_entry__
    __graft_entry__.build()


class Lin:
    """A quantized weight on the device and the oracle's codes, scales and zeros for it."""

    def __init__(self, K, N, bits, seed):
        W = inputs.weights(K, N, seed)
        codes, s, z = laq.laq_quantize_rtn(torch.from_numpy(W).cuda(), bits)
        self.packed = laq.laq_pack(codes, bits)
        self.s, self.z = s, z
        self.K, self.N, self.bits = K, N, bits
        self.ref = co.quantize_rtn(W, bits)


def nan_like(M, N):
    return torch.full((M, N), float("nan"), dtype=torch.float16, device="cuda")


def check_y(Y, X, lin):
    yref = co.gemm(np.asarray(X, np.float16), *lin.ref)
    err = np.abs(Y.cpu().numpy().astype(np.float64) - yref).max()
    assert err <= tolerance(yref), (err, tolerance(yref))
    return yref


@pytest.mark.parametrize("bits", [3, 4])
@pytest.mark.parametrize("M", [1, 2, 3, 4])
@pytest.mark.parametrize("K,N", [(128, 16), (384, 48), (1024, 1024), (2560, 1040), (9728, 2560)])
def test_single_entry(bits, M, K, N):
    lin = Lin(K, N, bits, seed=K + N + M + bits)
    X = inputs.activations(M, K, seed=M)
    Xd = torch.from_numpy(X).cuda()
    Y = nan_like(M, N)
    ws = laq.chain_workspace(1, "cuda")
    laq.laq_gemm_chain([(Xd, lin.packed, lin.s, lin.z, bits, Y, 1)], ws)
    assert laq.chain_status(ws) == 0
    check_y(Y, X, lin)
    # counters and per-CTA flags reset for the next call (the published parts may remain)
    zeroed = ((2 + 1 + 3) // 4 * 4 + 256) * 4
    assert int(ws[:zeroed].count_nonzero().item()) == 0


@pytest.mark.parametrize("bits", [3, 4])
@pytest.mark.parametrize("M", [1, 4])
def test_dependencies_and_stages(bits, M):
    """Entries in four stages: e0 | e1 e2 (both read Y0) | e3 (reads Y1) | e4 (reads Y3) e5
    (reads X0).  Stage sizes span 64..201 tiles, so CTAs hold one or two tiles each."""
    dims = [(512, 1024), (1024, 3200), (1024, 16), (3200, 768), (768, 128), (512, 2560)]
    lins = [Lin(K, N, bits, seed=100 + i) for i, (K, N) in enumerate(dims)]
    X0 = inputs.activations(M, 512, seed=7)
    X0d = torch.from_numpy(X0).cuda()
    Ys = [nan_like(M, N) for _, N in dims]
    src = [X0d, Ys[0], Ys[0], Ys[1], Ys[3], X0d]
    wait = [1, 1, 0, 1, 1, 0]
    ws = laq.chain_workspace(len(dims), "cuda")
    entries = [(src[i], lins[i].packed, lins[i].s, lins[i].z, bits, Ys[i], wait[i])
               for i in range(len(dims))]
    laq.laq_gemm_chain(entries, ws)
    assert laq.chain_status(ws) == 0
    # the oracle's chain, with its own fp16 intermediates
    r0 = check_y(Ys[0], X0, lins[0]).astype(np.float16)
    r1 = check_y(Ys[1], r0, lins[1]).astype(np.float16)
    check_y(Ys[2], r0, lins[2])
    r3 = check_y(Ys[3], r1, lins[3]).astype(np.float16)
    check_y(Ys[4], r3, lins[4])
    check_y(Ys[5], X0, lins[5])
    for Y in Ys:
        assert not torch.isnan(Y).any()


def test_repeated_calls_and_graph_replay():
    """The workspace comes back zeroed, so calls (and graph replays) follow one another."""
    bits, M = 3, 1
    lins = [Lin(2560, 4096, bits, 1), Lin(4096, 2560, bits, 2)]
    Xd = torch.empty((M, 2560), dtype=torch.float16, device="cuda")
    Y0, Y1 = nan_like(M, 4096), nan_like(M, 2560)
    spec = laq.Chain([(Xd, lins[0].packed, lins[0].s, lins[0].z, bits, Y0, 1),
                      (Y0, lins[1].packed, lins[1].s, lins[1].z, bits, Y1, 1)])
    ws = laq.chain_workspace(2, "cuda")

    def check(X):
        r0 = check_y(Y0, X, lins[0]).astype(np.float16)
        check_y(Y1, r0, lins[1])

    for seed in (1, 2, 3):
        X = inputs.activations(M, 2560, seed=seed)
        Xd.copy_(torch.from_numpy(X))
        spec.run(ws)
        assert laq.chain_status(ws) == 0
        check(X)
    s = torch.cuda.Stream()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, stream=s):
        spec.run(ws, stream=s)
    for seed in (4, 5):
        X = inputs.activations(M, 2560, seed=seed)
        Xd.copy_(torch.from_numpy(X))
        Y0.fill_(float("nan"))
        Y1.fill_(float("nan"))
        g.replay()
        assert laq.chain_status(ws) == 0
        check(X)


def test_recorded_error_stops_later_stages():
    """A status already recorded in the workspace makes every CTA give up at its first wait:
    the call returns promptly, later stages write nothing, the status word is kept for the
    host to read, and zeroing the workspace restores normal results.  (Stage 0 has no wait
    but its tiles that straddle two CTAs do, so its Y is only partly written.)"""
    bits, M = 3, 1
    lins = [Lin(1024, 1024, bits, 5), Lin(1024, 512, bits, 6)]
    X = inputs.activations(M, 1024, seed=9)
    Xd = torch.from_numpy(X).cuda()
    Y0, Y1 = nan_like(M, 1024), nan_like(M, 512)
    entries = [(Xd, lins[0].packed, lins[0].s, lins[0].z, bits, Y0, 1),
               (Y0, lins[1].packed, lins[1].s, lins[1].z, bits, Y1, 1)]
    ws = laq.chain_workspace(2, "cuda")
    ws[:4].view(torch.int32)[0] = 8                     # LAQ_ERR_TIMEOUT, as a timed-out wait
    laq.laq_gemm_chain(entries, ws)
    assert laq.chain_status(ws) == 8
    assert torch.isnan(Y1).all()
    ws.zero_()                                          # the documented recovery
    laq.laq_gemm_chain(entries, ws)
    assert laq.chain_status(ws) == 0
    r0 = check_y(Y0, X, lins[0]).astype(np.float16)
    check_y(Y1, r0, lins[1])


def test_rejects_stage_too_large_for_shared_memory():
    """A stage whose X (here 4 x 25600 fp16 = 200 KB) leaves no room for the weight ring."""
    bits, M = 3, 4
    lin = Lin(128 * 200, 16, bits, 1)
    X = torch.zeros((M, 128 * 200), dtype=torch.float16, device="cuda")
    Y = nan_like(M, 16)
    ws = laq.chain_workspace(1, "cuda")
    with pytest.raises(laq.LaqError) as ei:
        laq.laq_gemm_chain([(X, lin.packed, lin.s, lin.z, bits, Y, 1)], ws)
    assert ei.value.status == 4


@pytest.mark.parametrize("bits,M", [(3, 1), (4, 1), (3, 2), (4, 4)])
def test_qwen3_4b_layers_chain(bits, M):
    wp = WeightPass(model="qwen3-4b", bits=bits, M=M, layers=2, chain=True)
    assert wp.launches == 1
    g = wp.capture()
    wp.Ybuf.fill_(float("nan"))
    g.replay()
    torch.cuda.synchronize()
    assert laq.chain_status(wp.ws) == 0
    for idx in range(7):
        check_projection(wp, idx)
    _sampled(wp, layers={1})


def test_qwen3_4b_pass_chain_w3_m1():
    wp = WeightPass(model="qwen3-4b", bits=3, M=1, chain=True)
    g = wp.capture()
    wp.Ybuf.fill_(float("nan"))
    g.replay()
    torch.cuda.synchronize()
    assert laq.chain_status(wp.ws) == 0
    assert not torch.isnan(wp.Ybuf).any()
    _sampled(wp, layers={0, 17, 35})


def test_qwen3_8b_fused_pass_chain_w3_m1():
    wp = WeightPass(model="qwen3-8b", bits=3, M=1, outliers=True, fuse=True, chain=True)
    g = wp.capture()
    wp.Ybuf.fill_(float("nan"))
    g.replay()
    torch.cuda.synchronize()
    assert laq.chain_status(wp.ws) == 0
    _sampled(wp, layers={0, 35})


def test_stage_of_many_small_entries():
    """One stage of 20 entries with K = 128..640 and N = 16..80 (single-group and single-tile
    GEMVs, several X slots per CTA), then a stage reading one of their outputs, at M = 2."""
    bits, M = 4, 2
    rng = np.random.default_rng(3)
    dims = [(128 * int(rng.integers(1, 6)), 16 * int(rng.integers(1, 6))) for _ in range(20)]
    dims[7] = (dims[7][0], 128)   # its output is the last entry's X: K must be a multiple of 128
    lins = [Lin(K, N, bits, seed=300 + i) for i, (K, N) in enumerate(dims)]
    Xs = [inputs.activations(M, K, seed=400 + i) for i, (K, _) in enumerate(dims)]
    Xd = [torch.from_numpy(X).cuda() for X in Xs]
    Ys = [nan_like(M, N) for _, N in dims]
    last = Lin(dims[7][1], 48, bits, seed=399)
    Ylast = nan_like(M, 48)
    entries = [(Xd[i], lins[i].packed, lins[i].s, lins[i].z, bits, Ys[i], 1 if i == 0 else 0)
               for i in range(20)]
    entries.append((Ys[7], last.packed, last.s, last.z, bits, Ylast, 1))
    ws = laq.chain_workspace(len(entries), "cuda")
    laq.laq_gemm_chain(entries, ws)
    assert laq.chain_status(ws) == 0
    refs = [check_y(Ys[i], Xs[i], lins[i]) for i in range(20)]
    check_y(Ylast, refs[7].astype(np.float16), last)


def test_split_stage_with_tiles_straddling_entries():
    """Two entries of 80 tiles x 76 groups in one stage (160 tiles on the GPU's SMs: the stage
    is split by records, so tiles straddle CTAs, some next to the entry boundary)."""
    bits, M = 3, 1
    lins = [Lin(9728, 1280, bits, seed=500 + i) for i in range(2)]
    Xs = [inputs.activations(M, 9728, seed=510 + i) for i in range(2)]
    Ys = [nan_like(M, 1280) for _ in range(2)]
    entries = [(torch.from_numpy(Xs[i]).cuda(), lins[i].packed, lins[i].s, lins[i].z, bits,
                Ys[i], 1 if i == 0 else 0) for i in range(2)]
    ws = laq.chain_workspace(2, "cuda")
    for _ in range(2):     # twice: the published parts and flags are reused
        for Y in Ys:
            Y.fill_(float("nan"))
        laq.laq_gemm_chain(entries, ws)
        assert laq.chain_status(ws) == 0
        for i in range(2):
            check_y(Ys[i], Xs[i], lins[i])


def test_longest_chain():
    """LAQ_CHAIN_MAX entries of one record each (K = 128, N = 16) in 128 stages of three, through
    both the workspace and the static-scratch entry points: the longest parameter block, the
    most stage counters, and 152 CTAs of which most own no record of a stage."""
    bits, M = 3, 1
    n = laq._lib.CHAIN_MAX
    lins = [Lin(128, 16, bits, seed=600 + i) for i in range(3)]
    Xs = [inputs.activations(M, 128, seed=700 + i) for i in range(n)]
    Xd = [torch.from_numpy(X).cuda() for X in Xs]
    Ys = [nan_like(M, 16) for _ in range(n)]
    entries = [(Xd[i], lins[i % 3].packed, lins[i % 3].s, lins[i % 3].z, bits, Ys[i],
                1 if i % 3 == 0 else 0) for i in range(n)]
    spec = laq.Chain(entries)
    ws = laq.chain_workspace(n, "cuda")
    for run in (lambda: spec.run(ws), lambda: spec.run_static()):
        for Y in Ys:
            Y.fill_(float("nan"))
        run()
        torch.cuda.synchronize()
        assert all(not torch.isnan(Y).any() for Y in Ys)
        for i in range(0, n, 37):
            check_y(Ys[i], Xs[i], lins[i % 3])
    assert laq.chain_status(ws) == 0
