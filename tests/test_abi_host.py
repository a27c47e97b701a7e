"""Host-side checks of the C ABI (no GPU): the library loads, exports every symbol include/laq.h
declares, rejects invalid arguments with the documented status before touching a device, and
plans launches within the kernel's limits."""
import ctypes
import os
import re

import pytest

from tests.conftest import ROOT

import paper_2605_08755_gb300 as laq
from paper_2605_08755_gb300 import _lib, inputs

HEADER = os.path.join(ROOT, "include", "laq.h")


@pytest.fixture(scope="module")
def L():
    from paper_2605_08755_gb300 import build
    build.build()
    return _lib.lib()


def declared_functions():
    text = open(HEADER).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(laq_[a-z0-9_]+)\s*\(", text)))


def test_header_declares_the_abi():
    names = declared_functions()
    assert set(names) == set(_lib.EXPORTS)


def test_library_exports_every_declared_symbol(L):
    for name in declared_functions():
        assert hasattr(L, name), name


def test_status_strings_and_version(L):
    assert L.laq_version() == 1
    for code, name in _lib.STATUS.items():
        assert L.laq_status_str(code).decode().startswith(name)
    assert L.laq_status_str(12345)


def test_packed_bytes(L):
    assert laq.packed_bytes(2560, 4096, 3) == 2560 * 4096 * 3 // 8
    assert laq.packed_bytes(9728, 2560, 4) == 9728 * 2560 // 2
    assert laq.packed_bytes(100, 16, 3) == 0
    assert laq.packed_bytes(128, 16, 5) == 0
    assert laq.packed_bytes(0, 0, 3) == 0


FAKE = ctypes.c_void_p(0x10000)      # 16-byte aligned, never dereferenced: calls fail first
ODD = ctypes.c_void_p(0x10002)


def gemm(L, X=FAKE, M=1, K=256, N=32, packed=FAKE, s=FAKE, z=FAKE, bits=3, Y=FAKE):
    return L.laq_gemm_wxg128(X, M, K, N, packed, s, z, bits, Y, None)


def test_gemm_argument_validation(L):
    assert gemm(L, bits=2) == 2
    assert gemm(L, bits=5) == 2
    assert gemm(L, M=17) == 6
    assert gemm(L, M=-1) == 6
    assert gemm(L, K=100) == 4
    assert gemm(L, N=24) == 4
    assert gemm(L, K=-128) == 4
    assert gemm(L, X=None) == 1
    assert gemm(L, packed=None) == 1
    assert gemm(L, s=None) == 1
    assert gemm(L, z=None) == 1
    assert gemm(L, Y=None) == 1
    assert gemm(L, X=ODD) == 5
    assert gemm(L, Y=ODD) == 5
    assert gemm(L, packed=ODD) == 5
    assert gemm(L, s=ctypes.c_void_p(0x10001)) == 5
    assert gemm(L, s=ODD) == 5
    assert gemm(L, z=ctypes.c_void_p(0x10008)) == 5
    # empty problems are no-ops that never touch the device
    assert gemm(L, M=0) == 0
    assert gemm(L, N=0, Y=None) == 0


def test_gemm_config_validation(L):
    def run(**kw):
        base = dict(tiles_per_cta=1, warps=4, cluster=1, stages=4, pdl=0)
        base.update(kw)
        cfg = _lib.GemmConfig.make(**base)
        return L.laq_gemm_wxg128_config(FAKE, 1, 256, 32, FAKE, FAKE, FAKE, 3, FAKE,
                                        ctypes.byref(cfg), None)
    assert run(tiles_per_cta=3) == 9
    assert run(tiles_per_cta=16) == 9
    assert run(warps=0) == 9
    assert run(warps=17) == 9
    assert run(warps=16) == 9  # more than 8 warps only from M = 3 (this call has M = 1)
    assert run(cluster=3) == 9
    assert run(cluster=16) == 9
    assert run(stages=1) == 9
    assert run(stages=17) == 9
    assert run(pdl=2) == 9
    assert run(tiles_per_cta=2, warps=3) == 9
    assert run(tiles_per_cta=4, warps=2) == 9
    assert L.laq_gemm_wxg128_config(FAKE, 1, 256, 32, FAKE, FAKE, FAKE, 3, FAKE, None,
                                    None) == 1


def test_quantize_pack_argument_validation(L):
    q = L.laq_quantize_rtn
    assert q(FAKE, 256, 32, 3, 64, FAKE, FAKE, FAKE, None) == 3
    assert q(FAKE, 256, 32, 6, 128, FAKE, FAKE, FAKE, None) == 2
    assert q(FAKE, 200, 32, 3, 128, FAKE, FAKE, FAKE, None) == 4
    assert q(None, 256, 32, 3, 128, FAKE, FAKE, FAKE, None) == 1
    assert q(ctypes.c_void_p(0x10001), 256, 32, 3, 128, FAKE, FAKE, FAKE, None) == 5
    assert q(FAKE, 0, 32, 3, 128, None, None, None, None) == 0
    p = L.laq_pack
    assert p(FAKE, 256, 24, 3, FAKE, None) == 4
    assert p(FAKE, 256, 32, 3, ODD, None) == 5
    assert p(None, 256, 32, 3, FAKE, None) == 1
    assert p(FAKE, 0, 32, 3, None, None) == 0
    u = L.laq_unpack
    assert u(FAKE, 256, 32, 7, FAKE, None) == 2
    assert u(ODD, 256, 32, 3, FAKE, None) == 5


@pytest.mark.parametrize("bits", [3, 4])
@pytest.mark.parametrize("M", [1, 2, 3, 4, 5, 8, 9, 16])
def test_plan_is_valid_for_every_workload_shape(L, bits, M):
    shapes = {(K, N) for _, K, N in inputs.QWEN3_4B + inputs.QWEN3_8B}
    shapes |= {(1024, 1024), (128, 16), (256, 4096), (12288, 16)}
    for K, N in sorted(shapes):
        for sms in (152, 148, 1):
            c = laq.laq_gemm_plan(M, K, N, bits, sms)
            assert c.tiles_per_cta in (1, 2, 4, 8)
            assert 1 <= c.warps <= 16 and c.warps % c.tiles_per_cta == 0
            assert c.cluster in (1, 2, 4, 8) and c.cluster <= max(1, K // 128)
            assert 2 <= c.stages <= 16
            assert c.pdl == 0
            assert c.warps % c.tiles_per_cta == 0


def test_plan_rejects_bad_arguments(L):
    cfg = _lib.GemmConfig()
    assert L.laq_gemm_plan(1, 256, 32, 3, 0, ctypes.byref(cfg)) == 9
    assert L.laq_gemm_plan(1, 256, 32, 3, 152, None) == 1
    assert L.laq_gemm_plan(20, 256, 32, 3, 152, ctypes.byref(cfg)) == 6
    assert L.laq_gemm_plan(1, 250, 32, 3, 152, ctypes.byref(cfg)) == 4


def chain_entry(X=FAKE, packed=FAKE, s=FAKE, z=FAKE, Y=FAKE, M=1, K=256, N=32, bits=3, wait=1):
    return _lib.Gemv(X.value, packed.value, s.value, z.value, Y.value, M, K, N, bits, wait)


def chain(L, entries, ws=FAKE, ws_bytes=None, count=None):
    arr = (_lib.Gemv * max(1, len(entries)))(*entries)
    n = len(entries) if count is None else count
    if ws_bytes is None:
        ws_bytes = L.laq_chain_workspace_bytes(max(0, min(n, _lib.CHAIN_MAX)))
    return L.laq_gemm_chain(arr, n, ws, ws_bytes, None)


def test_chain_workspace_bytes(L):
    # counters (2 + count words, padded to 4) + 256 flags + 256 parts of 64 words, to 256 bytes
    def expect(n):
        words = (2 + n + 3) // 4 * 4 + 256 + 256 * 64
        return (words * 4 + 255) // 256 * 256
    assert L.laq_chain_workspace_bytes(0) == expect(0)
    assert L.laq_chain_workspace_bytes(252) == expect(252) == 67584
    assert L.laq_chain_workspace_bytes(_lib.CHAIN_MAX) == expect(_lib.CHAIN_MAX) == 68352
    assert L.laq_chain_workspace_bytes(_lib.CHAIN_MAX + 1) == 0
    assert L.laq_chain_workspace_bytes(-1) == 0


def test_chain_argument_validation(L):
    S = _lib.STATUS
    code = {v: k for k, v in S.items()}
    ok = chain_entry()
    assert chain(L, []) == 0                                         # nothing to do
    assert chain(L, [ok], count=_lib.CHAIN_MAX + 1) == code["LAQ_ERR_SHAPE"]
    assert L.laq_gemm_chain(None, 1, FAKE, 256, None) == code["LAQ_ERR_NULL"]
    assert chain(L, [ok], ws=ctypes.c_void_p(0)) == code["LAQ_ERR_WORKSPACE"]
    assert chain(L, [ok], ws=ODD) == code["LAQ_ERR_WORKSPACE"]
    assert chain(L, [ok] * 100, ws_bytes=256) == code["LAQ_ERR_WORKSPACE"]
    assert chain(L, [chain_entry(bits=5)]) == code["LAQ_ERR_BITS"]
    assert chain(L, [ok, chain_entry(bits=4)]) == code["LAQ_ERR_BITS"]
    assert chain(L, [chain_entry(M=0)]) == code["LAQ_ERR_M_RANGE"]
    assert chain(L, [chain_entry(M=5)]) == code["LAQ_ERR_M_RANGE"]
    assert chain(L, [ok, chain_entry(M=2)]) == code["LAQ_ERR_M_RANGE"]
    assert chain(L, [chain_entry(K=200)]) == code["LAQ_ERR_SHAPE"]
    assert chain(L, [chain_entry(N=40)]) == code["LAQ_ERR_SHAPE"]
    assert chain(L, [chain_entry(K=0)]) == code["LAQ_ERR_SHAPE"]
    assert chain(L, [chain_entry(N=0)]) == code["LAQ_ERR_SHAPE"]
    assert chain(L, [ok, chain_entry(Y=ctypes.c_void_p(0))]) == code["LAQ_ERR_NULL"]
    for field in ("X", "packed", "s", "z", "Y"):
        assert chain(L, [chain_entry(**{field: ODD})]) == code["LAQ_ERR_ALIGN"], field


def test_chain_static_argument_validation(L):
    code = {v: k for k, v in _lib.STATUS.items()}
    arr = (_lib.Gemv * 1)(chain_entry())
    assert L.laq_gemm_chain_static(arr, 0, None) == 0
    assert L.laq_gemm_chain_static(arr, _lib.CHAIN_MAX + 1, None) == code["LAQ_ERR_WORKSPACE"]
    assert L.laq_gemm_chain_static(arr, -1, None) == code["LAQ_ERR_SHAPE"]
    assert L.laq_gemm_chain_static(None, 1, None) == code["LAQ_ERR_NULL"]
    # every entry is checked before the static scratch is looked up or cleared: these return
    # without a device
    bad = (_lib.Gemv * 1)(chain_entry(bits=5))
    assert L.laq_gemm_chain_static(bad, 1, None) == code["LAQ_ERR_BITS"]
    bad = (_lib.Gemv * 1)(chain_entry(X=ODD))
    assert L.laq_gemm_chain_static(bad, 1, None) == code["LAQ_ERR_ALIGN"]
    bad = (_lib.Gemv * 1)(chain_entry(N=0))
    assert L.laq_gemm_chain_static(bad, 1, None) == code["LAQ_ERR_SHAPE"]


def test_plan_shares_x_across_tiles_above_m_two(L):
    one = lambda K, N, bits: laq.laq_gemm_plan(1, K, N, bits, 152).as_dict()
    shape = lambda c: (c.tiles_per_cta, c.warps, c.cluster, c.stages)
    for bits in (3, 4):
        for K, N in ((9728, 2560), (2560, 19456), (2560, 6144), (4096, 2560)):
            # M = 2: the M = 1 rule (the faster one there on GB300)
            assert laq.laq_gemm_plan(2, K, N, bits, 152).as_dict() == one(K, N, bits)
        for M in (3, 4):
            # the long-K down projection keeps the M = 1 shape (4-warp CTAs of 2 tiles, cluster 8)
            assert laq.laq_gemm_plan(M, 9728, 2560, bits, 152).as_dict() == one(9728, 2560, bits)
            # otherwise X shared by 4 tiles per CTA, K split until about one CTA per SM
            assert shape(laq.laq_gemm_plan(M, 2560, 6144, bits, 152))[:3] == (4, 8, 2)
            assert shape(laq.laq_gemm_plan(M, 4096, 2560, bits, 152))[:3] == (4, 8, 4)
            if (M, bits) != (4, 4):
                assert shape(laq.laq_gemm_plan(M, 2560, 19456, bits, 152)) == (4, 8, 1, 11)
    # gate|up at W4 M = 4: two 4-tile CTAs share an SM's 228 KB only with a shallower ring, so 8
    # tiles per CTA over a cluster of 2 (half the X per CTA), with the full ring
    assert shape(laq.laq_gemm_plan(4, 2560, 19456, 4, 152)) == (8, 8, 2, 11)
    # M > 4: 8 tiles per CTA, and a cluster K split towards one CTA per SM
    c = laq.laq_gemm_plan(8, 2560, 6144, 3, 152)
    assert (c.tiles_per_cta, c.warps, c.cluster) == (8, 8, 4)
    # M = 5..8, long K and fewer than 1.5 tiles per SM (down): 4-tile CTAs of 4 warps, cluster 8
    # (at W3 from M = 7; W3 M = 5, 6 keep 8-tile 8-warp CTAs)
    for M, bits in ((5, 4), (6, 4), (7, 3), (8, 3), (8, 4)):
        c = laq.laq_gemm_plan(M, 9728, 2560, bits, 152)
        assert (c.tiles_per_cta, c.warps, c.cluster) == (4, 4, 8), (M, bits)
    for M in (5, 6):
        c = laq.laq_gemm_plan(M, 9728, 2560, 3, 152)
        assert (c.tiles_per_cta, c.warps, c.cluster, c.stages) == (8, 8, 8, 11)
    # 16-warp CTAs (one per SM at a time) whose grid falls between one and two per SM: cluster 2
    c = laq.laq_gemm_plan(16, 4096, 24576, 3, 152)
    assert (c.tiles_per_cta, c.warps, c.cluster) == (8, 16, 2)
    # M > 4 where that leaves one 8-warp CTA per SM: 16-warp CTAs (two warps per tile); the
    # long-K down projection at M > 8 with half the cluster
    c = laq.laq_gemm_plan(8, 2560, 19456, 3, 152)
    assert (c.tiles_per_cta, c.warps, c.cluster) == (8, 16, 1)
    c = laq.laq_gemm_plan(16, 2560, 19456, 3, 152)
    assert (c.tiles_per_cta, c.warps, c.cluster) == (8, 16, 1)
    c = laq.laq_gemm_plan(16, 9728, 2560, 3, 152)
    assert (c.tiles_per_cta, c.warps, c.cluster) == (8, 16, 4)
    # 16 warps only from M = 3 (the M <= 2 kernels are built for at most 8)
    for M in (1, 2):
        for K, N in ((2560, 19456), (9728, 2560), (4096, 24576)):
            assert laq.laq_gemm_plan(M, K, N, 3, 152).warps <= 8
    # M = 1: the fused Qwen3-4B projections
    assert laq.laq_gemm_plan(1, 2560, 19456, 3, 152).tiles_per_cta == 4
    assert laq.laq_gemm_plan(1, 2560, 6144, 3, 152).tiles_per_cta == 2


def test_plan_of_the_decode_pass_projections(L):
    """The launch shapes (tiles per CTA, warps, cluster, ring stages) of the fused Qwen3-4B and
    Qwen3-8B projections at M = 1 on 152 SMs, each the best or within 1 % of the best of a
    sweep of every shape inside the pass on GB300."""
    shape = lambda M, K, N, b: tuple(laq.laq_gemm_plan(M, K, N, b, 152).as_dict()[k]
                                     for k in ("tiles_per_cta", "warps", "cluster", "stages"))
    for bits in (3, 4):
        for M in (1, 2):
            assert shape(M, 2560, 6144, bits) == (2, 8, 1, 6)      # q|k|v
            assert shape(M, 4096, 2560, bits) == (1, 8, 1, 5)      # o
            assert shape(M, 2560, 19456, bits) == (4, 8, 1, 11)    # gate|up
            assert shape(M, 9728, 2560, bits) == (2, 4, 8, 6)      # down
        assert shape(1, 4096, 6144, bits) == (2, 8, 1, 9)
        assert shape(1, 4096, 4096, bits) == (1, 8, 1, 5)
        # 1536 tiles: 2-tile CTAs in three waves, not one wave of 8-tile CTAs
        assert shape(1, 4096, 24576, bits) == (2, 8, 1, 9)
        # 256 tiles (1.7 per SM): no cluster; at W4 the ring gives up stages so that two CTAs
        # share an SM
        assert shape(1, 12288, 4096, bits) == (1, 8, 1, 13 if bits == 3 else 10)


@pytest.mark.parametrize("bits", [3, 4])
def test_plan_splits_k_of_narrow_outputs_at_m_one(L, bits):
    # Fewer than 1.5 16-column tiles per SM and a K long enough that 8-warp CTAs would leave a
    # warp more than 5 records: 4-warp CTAs of 2 tiles, K split over a cluster until a warp
    # holds at most 5 records and the grid covers every SM.
    for K, N, cl in ((9728, 2560, 8),):
        c = laq.laq_gemm_plan(1, K, N, bits, 152)
        assert (c.tiles_per_cta, c.warps, c.cluster) == (2, 4, cl), (K, N, c.as_dict())
        per_warp = c.tiles_per_cta * -(-(K // 128) // c.cluster) / c.warps
        assert per_warp <= 5 or c.cluster == 8
        assert (N // 16 + 1) // 2 * c.cluster >= 152 or c.cluster == 8
    # shorter K (o, q, k, v of Qwen3-4B) and wide outputs keep 8-warp CTAs
    for K, N in ((4096, 2560), (2560, 4096), (2560, 1024), (2560, 19456), (2560, 6144)):
        assert laq.laq_gemm_plan(1, K, N, bits, 152).warps >= 5, (K, N)


def test_gemm_prologue_argument_validation(L):
    def run(kind=1, eps=1e-6, R=None, R_out=None, w=FAKE, X=FAKE):
        pro = _lib.GemmPrologue(kind, eps, R, R_out, w)
        return L.laq_gemm_wxg128_prologue(X, 1, 256, 32, FAKE, FAKE, FAKE, 3, FAKE,
                                          ctypes.byref(pro), None, None)
    assert run(kind=3) == 9             # unknown kind: LAQ_ERR_CONFIG
    assert run(kind=-1) == 9
    assert run(w=None) == 1             # RMSNorm without weights
    assert run(eps=-1.0) == 4
    assert run(eps=float("nan")) == 4
    assert run(R=FAKE, R_out=FAKE) == 4          # R_out may not alias R ...
    assert run(R_out=FAKE) == 4                  # ... nor X (both FAKE here)
    assert run(w=ODD) == 5
    assert run(R=ODD) == 5
    assert run(R_out=ctypes.c_void_p(0x20008)) == 5
    assert run(kind=2, X=ODD) == 5


def test_rotation_argument_validation(L):
    def rot(X=FAKE, M=1, K=256, alpha=None, pairs=FAKE, cs=FAKE, rounds=4, Y=FAKE):
        return L.laq_pairwise_rotate(X, M, K, alpha, pairs, cs, rounds, Y, None)
    assert rot(M=0) == 0                # nothing to do, no launch
    assert rot(X=None) == 1
    assert rot(Y=None) == 1
    assert rot(pairs=None) == 1
    assert rot(cs=None) == 1
    assert rot(K=200) == 4
    assert rot(K=0) == 4
    assert rot(M=65536) == 4
    assert rot(M=-1) == 4
    assert rot(rounds=17) == 4
    assert rot(rounds=-1) == 4
    assert rot(X=ODD) == 5
    assert rot(Y=ctypes.c_void_p(0x10008)) == 5
    assert rot(alpha=ODD) == 5
    assert rot(pairs=ctypes.c_void_p(0x10008)) == 5
    tables = L.laq_rotation_tables
    assert tables(None, 0, None, None) == 0
    assert tables(None, 5, FAKE, None) == 1
    assert tables(FAKE, 5, None, None) == 1
    assert tables(FAKE, -1, FAKE, None) == 4
    assert tables(FAKE, (1 << 31) + 1, FAKE, None) == 4
    assert tables(ctypes.c_void_p(0x10002), 5, FAKE, None) == 5
    assert tables(FAKE, 5, ctypes.c_void_p(0x10004), None) == 5
