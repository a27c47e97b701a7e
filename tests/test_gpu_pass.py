"""The planned pass (laq_pass_plan_build, laq_pass_prepare, laq_pass_run) against the oracle.

Every entry's Y must satisfy the GEMV tolerance against the oracle's fp64 product of the oracle's
own codes, scales and zeros; chains with dependencies feed one entry's Y to the next entry as X,
every Y pre-filled with NaN.
"""
import numpy as np
import pytest
import torch

import paper_2605_08755_gb300 as laq
from paper_2605_08755_gb300 import _lib, inputs
from paper_2605_08755_gb300.weight_pass import WeightPass
from tests.test_gpu_chain import Lin, check_y, nan_like
from tests.test_gpu_workloads import _sampled, check_projection

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def built():
    import __graft_entry__
    __graft_entry__.build()


def run(entries):
    plan = _lib.PassPlan(entries, "cuda")
    plan.run()
    assert plan.status() == 0
    # a completed call leaves the workspace zero for the next one
    assert int(plan.ws.count_nonzero().item()) == 0
    return plan


@pytest.mark.parametrize("bits", [3, 4])
@pytest.mark.parametrize("M", [1, 2, 3, 4])
@pytest.mark.parametrize("K,N", [(128, 16), (384, 48), (1024, 1024), (2560, 1040),
                                 (9728, 2560), (13312, 32)])
def test_single_entry(bits, M, K, N):
    lin = Lin(K, N, bits, seed=K + N + bits)
    X = inputs.activations(M, K, seed=K + M)
    Y = nan_like(M, N)
    run([(torch.from_numpy(X).cuda(), lin.packed, lin.s, lin.z, bits, Y, 1)])
    check_y(Y, X, lin)


@pytest.mark.parametrize("bits,M", [(3, 1), (4, 1), (3, 2), (4, 4)])
def test_dependencies_and_stages(bits, M):
    """e0 | e1 e2 (both read Y0) | e3 (reads Y1) | e4 (reads Y3) e5 (reads X0)."""
    dims = [(512, 1024), (1024, 3200), (1024, 16), (3200, 768), (768, 128), (512, 2560)]
    lins = [Lin(K, N, bits, seed=100 + i) for i, (K, N) in enumerate(dims)]
    X0 = inputs.activations(M, 512, seed=7)
    X0d = torch.from_numpy(X0).cuda()
    Ys = [nan_like(M, N) for _, N in dims]
    src = [X0d, Ys[0], Ys[0], Ys[1], Ys[3], X0d]
    wait = [1, 1, 0, 1, 1, 0]
    run([(src[i], lins[i].packed, lins[i].s, lins[i].z, bits, Ys[i], wait[i])
         for i in range(len(dims))])
    r0 = check_y(Ys[0], X0, lins[0]).astype(np.float16)
    r1 = check_y(Ys[1], r0, lins[1]).astype(np.float16)
    check_y(Ys[2], r0, lins[2])
    r3 = check_y(Ys[3], r1, lins[3]).astype(np.float16)
    check_y(Ys[4], r3, lins[4])
    check_y(Ys[5], X0, lins[5])


def test_repeated_calls_deterministic_and_graph_replay():
    bits = 3
    lins = [Lin(2560, 4096, bits, 1), Lin(4096, 2560, bits, 2)]
    Xd = torch.empty((1, 2560), dtype=torch.float16, device="cuda")
    Y0, Y1 = nan_like(1, 4096), nan_like(1, 2560)
    plan = _lib.PassPlan([(Xd, lins[0].packed, lins[0].s, lins[0].z, bits, Y0, 1),
                          (Y0, lins[1].packed, lins[1].s, lins[1].z, bits, Y1, 1)], "cuda")
    X = inputs.activations(1, 2560, seed=1)
    Xd.copy_(torch.from_numpy(X))
    outs = []
    for _ in range(3):
        Y0.fill_(float("nan"))
        Y1.fill_(float("nan"))
        plan.run()
        assert plan.status() == 0
        outs.append((Y0.clone(), Y1.clone()))
    for a, b in outs[1:]:
        assert torch.equal(a, outs[0][0]) and torch.equal(b, outs[0][1])
    r0 = check_y(Y0, X, lins[0]).astype(np.float16)
    check_y(Y1, r0, lins[1])
    s = torch.cuda.Stream()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, stream=s):
        plan.run(stream=s)
    for seed in (4, 5):
        X = inputs.activations(1, 2560, seed=seed)
        Xd.copy_(torch.from_numpy(X))
        Y0.fill_(float("nan"))
        Y1.fill_(float("nan"))
        g.replay()
        assert plan.status() == 0
        r0 = check_y(Y0, X, lins[0]).astype(np.float16)
        check_y(Y1, r0, lins[1])


def test_recorded_error_stops_later_stages():
    """A status already in the workspace makes every CTA give up at its first stage wait: the
    call returns, the second stage writes nothing, the status stays; zeroing the workspace (the
    documented recovery) restores normal results."""
    bits = 3
    lins = [Lin(1024, 1024, bits, 5), Lin(1024, 512, bits, 6)]
    X = inputs.activations(1, 1024, seed=9)
    Xd = torch.from_numpy(X).cuda()
    Y0, Y1 = nan_like(1, 1024), nan_like(1, 512)
    plan = _lib.PassPlan([(Xd, lins[0].packed, lins[0].s, lins[0].z, bits, Y0, 1),
                          (Y0, lins[1].packed, lins[1].s, lins[1].z, bits, Y1, 1)], "cuda")
    plan.ws[:4].view(torch.int32)[0] = 8            # LAQ_ERR_TIMEOUT, as a timed-out wait
    plan.run()
    assert plan.status() == 8
    assert torch.isnan(Y1).all()
    plan.ws.zero_()
    plan.run()
    assert plan.status() == 0
    r0 = check_y(Y0, X, lins[0]).astype(np.float16)
    check_y(Y1, r0, lins[1])


def test_plan_for_another_sm_count_is_rejected():
    bits = 3
    lin = Lin(256, 32, bits, 3)
    Xd = torch.from_numpy(inputs.activations(1, 256, seed=3)).cuda()
    Y = nan_like(1, 32)
    chain = _lib.Chain([(Xd, lin.packed, lin.s, lin.z, bits, Y, 1)])
    sms = torch.cuda.get_device_properties(0).multi_processor_count
    plan, dev_bytes = _lib.pass_plan(chain.array, 1, sms - 1)
    buf = torch.empty((dev_bytes,), dtype=torch.uint8, device="cuda")
    nws = int(_lib.lib().laq_pass_workspace_bytes(plan))
    ws = torch.zeros((nws,), dtype=torch.uint8, device="cuda")
    st = _lib.lib().laq_pass_run(plan, _lib._ptr(buf), _lib._ptr(ws), nws, _lib._stream(None))
    assert st == 9                                  # LAQ_ERR_CONFIG, nothing launched


def test_stage_of_many_small_entries():
    """One stage of 20 entries with K = 128..640 and N = 16..80, then one reading an output."""
    bits = 4
    rng = np.random.default_rng(3)
    dims = [(128 * int(rng.integers(1, 6)), 16 * int(rng.integers(1, 6))) for _ in range(20)]
    dims[7] = (dims[7][0], 128)
    lins = [Lin(K, N, bits, seed=300 + i) for i, (K, N) in enumerate(dims)]
    Xs = [inputs.activations(1, K, seed=400 + i) for i, (K, _) in enumerate(dims)]
    Ys = [nan_like(1, N) for _, N in dims]
    last = Lin(dims[7][1], 48, bits, seed=399)
    Ylast = nan_like(1, 48)
    entries = [(torch.from_numpy(Xs[i]).cuda(), lins[i].packed, lins[i].s, lins[i].z, bits,
                Ys[i], 1 if i == 0 else 0) for i in range(20)]
    entries.append((Ys[7], last.packed, last.s, last.z, bits, Ylast, 1))
    run(entries)
    refs = [check_y(Ys[i], Xs[i], lins[i]) for i in range(20)]
    check_y(Ylast, refs[7].astype(np.float16), last)


def test_longest_chain():
    """LAQ_CHAIN_MAX entries of one record each in 128 stages of three: most SMs own no record
    of a stage."""
    bits = 3
    n = laq._lib.CHAIN_MAX
    lins = [Lin(128, 16, bits, seed=600 + i) for i in range(3)]
    Xs = [inputs.activations(1, 128, seed=700 + i) for i in range(n)]
    Ys = [nan_like(1, 16) for _ in range(n)]
    run([(torch.from_numpy(Xs[i]).cuda(), lins[i % 3].packed, lins[i % 3].s, lins[i % 3].z,
          bits, Ys[i], 1 if i % 3 == 0 else 0) for i in range(n)])
    for i in range(0, n, 37):
        check_y(Ys[i], Xs[i], lins[i % 3])


@pytest.mark.parametrize("bits,fuse,M", [(3, True, 1), (4, True, 1), (3, False, 1),
                                         (3, True, 2), (4, True, 4)])
def test_qwen3_4b_pass_planned(bits, fuse, M):
    wp = WeightPass(model="qwen3-4b", bits=bits, M=M, fuse=fuse, planned=True)
    assert wp.launches == 1
    g = wp.capture()
    wp.Ybuf.fill_(float("nan"))
    g.replay()
    torch.cuda.synchronize()
    assert wp.plan.status() == 0
    assert not torch.isnan(wp.Ybuf).any()
    _sampled(wp, layers={0, 17, 35})


def test_qwen3_4b_layers_planned_fully():
    wp = WeightPass(model="qwen3-4b", bits=3, M=1, layers=2, fuse=True, planned=True)
    wp.Ybuf.fill_(float("nan"))
    wp.run()
    torch.cuda.synchronize()
    assert wp.plan.status() == 0
    for idx in range(len(wp.linears)):
        check_projection(wp, idx)


def test_qwen3_8b_fused_pass_planned():
    wp = WeightPass(model="qwen3-8b", bits=3, M=1, outliers=True, fuse=True, planned=True)
    g = wp.capture()
    wp.Ybuf.fill_(float("nan"))
    g.replay()
    torch.cuda.synchronize()
    assert wp.plan.status() == 0
    _sampled(wp, layers={0, 35})


@pytest.mark.parametrize("bits,M", [(3, 1), (4, 2)])
def test_prepared_buffer_bit_exact(bits, M):
    """laq_pass_prepare's output byte for byte: every stream record is its entry's packed record
    followed by the scale/zero row pairs of its (group, tile), in the plan's order, and the
    tables are the plan's."""
    from tests.test_pass_lanes import stream_sz
    from tests.test_pass_plan import parse
    dims = [(384, 48), (1024, 160), (256, 16)]
    lins = [Lin(K, N, bits, seed=40 + i) for i, (K, N) in enumerate(dims)]
    Xs = [torch.from_numpy(inputs.activations(M, K, seed=i)).cuda()
          for i, (K, _) in enumerate(dims)]
    Ys = [nan_like(M, N) for _, N in dims]
    plan = _lib.PassPlan([(Xs[i], lins[i].packed, lins[i].s, lins[i].z, bits, Ys[i], i % 2)
                          for i in range(3)], "cuda")
    torch.cuda.synchronize()
    tb = parse(plan.plan)
    h = tb["h"]
    buf = plan.buffer.cpu().numpy()
    rb, rbc = int(h["rb"]), int(h["rb"]) - 48
    host = np.frombuffer(plan.plan, dtype=np.uint8)
    tables = host[int(h["tables_h"]):int(h["tables_h"] + h["tables_bytes"])]
    s0 = int(h["stream_bytes"])
    assert np.array_equal(buf[s0:s0 + tables.size], tables)
    packed = [l.packed.cpu().numpy() for l in lins]
    s16 = [l.s.cpu().numpy().view(np.uint16) for l in lins]
    z8 = [l.z.cpu().numpy() for l in lins]
    for i, gr in enumerate(tb["gather"]):
        e, rid = int(gr["e"]), int(gr["rid"])
        G = dims[e][0] // 128
        t, g = divmod(rid, G)
        rec = buf[i * rb:(i + 1) * rb]
        assert np.array_equal(rec[:rbc], packed[e][rid * rbc:(rid + 1) * rbc]), i
        sw, zw = stream_sz(s16[e][g, 16 * t:16 * t + 16].view(np.float16),
                           z8[e][g, 16 * t:16 * t + 16])
        assert list(rec[rbc:rbc + 32].view("<u4")) == sw, i
        assert list(rec[rbc + 32:rbc + 48].view("<u2")) == zw, i
