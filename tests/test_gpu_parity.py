"""GPU vs oracle parity through the C ABI: quantizer, packing and the GEMV / skinny GEMM.

Codes, scales, zeros and packed words must be bit-exact; Y must satisfy
|Y_gpu - Y_ref| <= 5e-3 * max|Y_ref| + 1e-3 per element (tests.conftest.tolerance), with the
oracle's fp64 Y as reference.  Sizes span several tiles, several groups and ragged tails.
"""
import ctypes
import itertools

import numpy as np
import pytest
import torch

import paper_2605_08755_gb300 as laq
from oracle import c_oracle as co
from paper_2605_08755_gb300 import inputs
from tests.conftest import tolerance
from tests.test_oracle_pins import _load_ties, _planted

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def built():
    from paper_2605_08755_gb300 import build
    build.build()
    laq.lib()


def dev(a):
    return torch.from_numpy(np.ascontiguousarray(a)).cuda()


def gpu_quantize(W, bits):
    codes, s, z = laq.laq_quantize_rtn(dev(W), bits)
    torch.cuda.synchronize()
    return codes.cpu().numpy(), s.cpu().numpy(), z.cpu().numpy()


def assert_quant_equal(got, ref):
    gc, gs, gz = got
    rc, rs, rz = ref
    assert np.array_equal(gs.view(np.uint16), np.asarray(rs).view(np.uint16))
    assert np.array_equal(gz, rz)
    assert np.array_equal(gc, rc)


@pytest.mark.parametrize("bits", [3, 4])
@pytest.mark.parametrize("K,N,outliers", [(1024, 1024, False), (384, 48, True), (128, 16, False),
                                          (2560, 1040, False), (256, 2000, True)])
def test_quantize_bit_exact(bits, K, N, outliers):
    W = inputs.weights(K, N, seed=K + N + bits, outliers=outliers)
    assert_quant_equal(gpu_quantize(W, bits), co.quantize_rtn(W, bits))


@pytest.mark.parametrize("bits", [3, 4])
def test_quantize_special_groups(bits):
    # planted codes (closed-form s, z, q), constant groups, ties and tiny ranges in one matrix
    Wp, Q, s0, z0 = _planted(bits, G=2, N=16, seed=1, m=3, e=9)
    consts = np.zeros((256, 16), np.float16)
    for i, c in enumerate([0.013, -0.013, 0.0, -0.0, 65504.0, -65504.0, 2.0 ** -20,
                           -(2.0 ** -24), 1.0, -3.5, 7.0, -1e-3, 0.25, -0.25, 3e-5, 100.0]):
        consts[:, i] = c
    ties = np.zeros((256, 16), np.float16)
    for col, blk in enumerate(b for b in _load_ties() if b["bits"] == bits):
        for r, (w, _) in enumerate(blk["w"]):
            ties[r, col] = w
    ties[128:, 5] = np.float16(2.0 ** -24) * np.arange(128).astype(np.float16)
    W = np.concatenate([Wp, consts, ties], axis=1)
    got = gpu_quantize(W, bits)
    assert_quant_equal(got, co.quantize_rtn(W, bits))
    assert np.array_equal(got[0][:, :16], Q)
    Wh = co.dequant(*got)
    assert np.array_equal(Wh[:, 16:32], consts.astype(np.float64))


@pytest.mark.parametrize("bits", [3, 4])
@pytest.mark.parametrize("K,N", [(128, 16), (384, 48), (1024, 1024), (2560, 96)])
def test_pack_and_unpack_bit_exact(bits, K, N):
    rng = np.random.default_rng(K * N + bits)
    codes = rng.integers(0, 1 << bits, size=(K, N)).astype(np.uint8)
    packed = laq.laq_pack(dev(codes), bits)
    ref = co.pack(codes, bits)
    assert np.array_equal(packed.cpu().numpy().view(np.uint32), ref)
    back = laq.laq_unpack(dev(ref.view(np.uint8)), K, N, bits)
    assert np.array_equal(back.cpu().numpy(), codes)


def prepare(K, N, bits, seed, outliers=False):
    W = inputs.weights(K, N, seed=seed, outliers=outliers)
    codes, s, z = co.quantize_rtn(W, bits)
    packed = dev(co.pack(codes, bits).view(np.uint8))
    return codes, s, z, packed, dev(s.view(np.uint16)).view(torch.float16), dev(z)


def run_gemm(X, packed, s_d, z_d, bits, config=None):
    Y = laq.laq_gemm_wxg128(dev(X), packed, s_d, z_d, bits, config=config)
    torch.cuda.synchronize()
    return Y.cpu().numpy().astype(np.float64)


def check_y(y, yref):
    err = np.abs(y - yref)
    tol = tolerance(yref)
    assert err.max() <= tol, f"max err {err.max()} > tol {tol}"


@pytest.mark.parametrize("bits", [3, 4])
@pytest.mark.parametrize("M", list(range(1, 17)))
def test_gemm_parity_all_m(bits, M):
    K, N = 1280, 272    # 10 groups, 17 tiles: ragged against every tile / warp / cluster split
    codes, s, z, packed, s_d, z_d = prepare(K, N, bits, seed=M)
    X = inputs.activations(M, K, seed=M)
    check_y(run_gemm(X, packed, s_d, z_d, bits), co.gemm(X, codes, s, z))


@pytest.mark.parametrize("bits", [3, 4])
@pytest.mark.parametrize("M,K,N", [(1, 1024, 1024), (1, 128, 16), (2, 9728, 64),
                                   (1, 2560, 1040), (16, 4096, 48), (5, 384, 4096)])
def test_gemm_parity_shapes(bits, M, K, N):
    codes, s, z, packed, s_d, z_d = prepare(K, N, bits, seed=K + N)
    X = inputs.activations(M, K, seed=K)
    check_y(run_gemm(X, packed, s_d, z_d, bits), co.gemm(X, codes, s, z))


CONFIGS = [laq.GemmConfig.make(nt, w, cl, st, pdl)
           for nt, w, cl, st, pdl in itertools.product((1, 2, 4, 8), (1, 2, 3, 4, 8, 12, 16),
                                                       (1, 2, 4, 8), (2, 3, 16), (0, 1))]


SMEM_OPTIN = 232448   # bytes of dynamic shared memory a CTA may opt into on sm_100 / sm_103


def smem_needed(M, K, bits, cfg):
    """Mirror of the library's shared-memory budget: per-warp cp.async rings, staged X with its
    group sums (about 64 KB per phase; padded rows from M = 3), the zero block (M <= 2), scales
    and zeros, per-CTA partial sums."""
    rec = 1024 if bits == 4 else 768
    gc = -(-(K // 128) // cfg.cluster)
    mp = 1 if M <= 1 else 2 if M <= 2 else 4 if M <= 4 else 8 if M <= 8 else 16
    padded = mp >= 4
    per_group = M * ((17 if padded else 16) * 16 + 8)
    gpp = max(1, min(gc, 64 * 1024 // per_group))
    # X rows in 16-byte chunks (padded: 17 per group, row stride 2 mod 8), zero block if not
    row_chunks = gpp * 17 + (2 - gpp * 17) % 8 if padded else gpp * 16
    return (cfg.warps * cfg.stages * rec + M * row_chunks * 16 + M * gpp * 8
            + (0 if padded else 64) + gc * cfg.tiles_per_cta * 48 + cfg.tiles_per_cta * mp * 64)


@pytest.mark.parametrize("bits", [3, 4])
@pytest.mark.parametrize("M", [1, 3, 8, 11])
def test_gemm_every_launch_configuration(bits, M):
    K, N = 1280, 80     # G = 10 groups, T = 5 tiles
    codes, s, z, packed, s_d, z_d = prepare(K, N, bits, seed=7 * M)
    X = inputs.activations(M, K, seed=3 * M)
    yref = co.gemm(X, codes, s, z)
    for cfg in CONFIGS:
        if cfg.warps % cfg.tiles_per_cta or (cfg.warps > 8 and M < 3):
            with pytest.raises(laq.LaqError) as e:
                run_gemm(X, packed, s_d, z_d, bits, config=cfg)
            assert e.value.status == 9
            continue
        if smem_needed(M, K, bits, cfg) > SMEM_OPTIN:
            with pytest.raises(laq.LaqError) as e:
                run_gemm(X, packed, s_d, z_d, bits, config=cfg)
            assert e.value.status == 9
            continue
        check_y(run_gemm(X, packed, s_d, z_d, bits, config=cfg), yref)


def test_gemm_cluster_larger_than_groups():
    # cluster of 8 CTAs over 2 groups: six CTAs own no group and contribute zeros
    codes, s, z, packed, s_d, z_d = prepare(256, 32, 3, seed=2)
    X = inputs.activations(2, 256, seed=2)
    cfg = laq.GemmConfig.make(1, 4, 8, 3, 0)
    check_y(run_gemm(X, packed, s_d, z_d, 3, config=cfg), co.gemm(X, codes, s, z))


@pytest.mark.parametrize("bits", [3, 4])
def test_gemm_exact_for_small_integers(bits):
    """Small-integer X and power-of-two scales make every product and sum exact in fp32, so
    the fp16 output must equal the oracle's exact Y rounded once to fp16, bit for bit."""
    W, Q, s0, z0 = _planted(bits, G=4, N=48, seed=5, m=1, e=5)
    codes, s, z = co.quantize_rtn(W, bits)
    assert np.array_equal(codes, Q)
    rng = np.random.default_rng(5)
    for M in (1, 4, 16):
        X = rng.integers(-3, 4, size=(M, 512)).astype(np.float16)
        Y = laq.laq_gemm_wxg128(dev(X), dev(co.pack(codes, bits).view(np.uint8)),
                                dev(s.view(np.uint16)).view(torch.float16), dev(z), bits)
        torch.cuda.synchronize()
        yref = co.gemm(X, codes, s, z).astype(np.float16)
        assert np.array_equal(Y.cpu().numpy().view(np.uint16), yref.view(np.uint16))


def test_gemm_one_hot_rows():
    codes, s, z, packed, s_d, z_d = prepare(512, 64, 3, seed=9)
    What = co.dequant(codes, s, z)
    X = np.zeros((16, 512), np.float16)
    rows = [0, 1, 7, 8, 127, 128, 200, 255, 256, 300, 383, 384, 400, 450, 510, 511]
    for m, k in enumerate(rows):
        X[m, k] = 1.0
    y = run_gemm(X, packed, s_d, z_d, 3)
    assert np.array_equal(y, What[rows].astype(np.float16).astype(np.float64))


def test_gemm_deterministic():
    codes, s, z, packed, s_d, z_d = prepare(2560, 1024, 3, seed=4)
    X = dev(inputs.activations(3, 2560, seed=4))
    a = laq.laq_gemm_wxg128(X, packed, s_d, z_d, 3).clone()
    b = laq.laq_gemm_wxg128(X, packed, s_d, z_d, 3)
    torch.cuda.synchronize()
    assert torch.equal(a.view(torch.int16), b.view(torch.int16))


def _p(t):
    return ctypes.c_void_p(t.data_ptr())


def test_gemm_empty_shapes():
    codes, s, z, packed, s_d, z_d = prepare(128, 16, 3, seed=1)
    X = dev(inputs.activations(2, 128, seed=1))
    Y = torch.full((2, 16), 7.0, dtype=torch.float16, device="cuda")
    # K = 0: Y := 0
    assert laq.lib().laq_gemm_wxg128(None, 2, 0, 16, None, None, None, 3, _p(Y), None) == 0
    torch.cuda.synchronize()
    assert torch.count_nonzero(Y).item() == 0
    # M = 0 and N = 0 are no-ops
    Y.fill_(7.0)
    st = laq.lib().laq_gemm_wxg128(_p(X), 0, 128, 16, _p(packed), _p(s_d), _p(z_d), 3, _p(Y),
                                   None)
    st2 = laq.lib().laq_gemm_wxg128(_p(X), 2, 128, 0, _p(packed), _p(s_d), _p(z_d), 3, _p(Y),
                                    None)
    torch.cuda.synchronize()
    assert st == 0 and st2 == 0 and torch.all(Y == 7.0)


def test_gemm_rejects_misaligned_device_pointers():
    codes, s, z, packed, s_d, z_d = prepare(128, 16, 3, seed=1)
    X = dev(inputs.activations(1, 136, seed=1))
    X_off = X.view(-1)[4:132].view(1, 128)       # 8 bytes past a 16-byte boundary
    with pytest.raises(laq.LaqError) as e:
        laq.laq_gemm_wxg128(X_off, packed, s_d, z_d, 3)
    assert e.value.status == 5


def test_graph_capture_and_replay():
    cases = [(1, 1024, 1024, 3), (4, 2560, 96, 4), (16, 384, 4096, 3)]
    mats = [prepare(K, N, b, seed=K + b) for _, K, N, b in cases]
    Xs = [dev(inputs.activations(M, K, seed=K)) for M, K, _, _ in cases]
    eager = [laq.laq_gemm_wxg128(X, m[3], m[4], m[5], c[3]) for X, m, c in zip(Xs, mats, cases)]
    Ys = [torch.empty_like(y) for y in eager]
    g = torch.cuda.CUDAGraph()
    s = torch.cuda.Stream()
    with torch.cuda.graph(g, stream=s):
        for X, m, c, Y in zip(Xs, mats, cases, Ys):
            laq.laq_gemm_wxg128(X, m[3], m[4], m[5], c[3], Y=Y, stream=s)
    for _ in range(2):
        for Y in Ys:
            Y.zero_()
        g.replay()
        torch.cuda.synchronize()
        for a, b_ in zip(eager, Ys):
            assert torch.equal(a.view(torch.int16), b_.view(torch.int16))


def test_pdl_chain_respects_the_data_dependency():
    """A chain where each GEMV's input is the previous GEMV's output, launched with programmatic
    dependent launch: results must equal the plain stream-ordered chain."""
    K = N = 1024
    mats = [prepare(K, N, 3, seed=100 + i) for i in range(6)]
    x0 = dev(inputs.activations(1, K, seed=3))
    cfg = laq.laq_gemm_plan(1, K, N, 3, torch.cuda.get_device_properties(0).multi_processor_count)
    pdl = laq.GemmConfig.make(cfg.tiles_per_cta, cfg.warps, cfg.cluster, cfg.stages, 1)

    def chain(config):
        x = x0
        for m in mats:   # back-to-back library launches: the next reads what the last wrote
            x = laq.laq_gemm_wxg128(x, m[3], m[4], m[5], 3, config=config)
        torch.cuda.synchronize()
        return x

    ref = chain(None)
    for _ in range(3):
        assert torch.equal(chain(pdl).view(torch.int16), ref.view(torch.int16))
