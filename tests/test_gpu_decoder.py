"""GPU parity of the decoder operations around the projections (include/laq.h, laq_decode.cu)
and of a whole decode step, against oracle/decoder.py.  Tolerance per element, as for Y:
|gpu - ref| <= 5e-3 * max|ref| + 1e-3."""
import math

import numpy as np
import pytest

torch = pytest.importorskip("torch")

import paper_2605_08755_gb300 as laq  # noqa: E402
from paper_2605_08755_gb300 import _lib, inputs  # noqa: E402
from oracle import decoder as dec  # noqa: E402

pytestmark = pytest.mark.gpu
DEV = "cuda"
RNG = np.random.default_rng(77)


def f16(a):
    return np.asarray(a, np.float64).astype(np.float16)


def dev(a):
    return torch.from_numpy(np.ascontiguousarray(a)).to(DEV)


def host(t):
    torch.cuda.synchronize()
    return t.cpu().numpy()


def close(gpu, ref, what=""):
    g, r = np.asarray(gpu, np.float64), np.asarray(ref, np.float64)
    tol = 5e-3 * np.abs(r).max() + 1e-3
    err = np.abs(g - r).max()
    assert err <= tol, f"{what}: max err {err} > tol {tol}"


# ---- RMSNorm ----

@pytest.mark.parametrize("M,H", [(1, 2560), (3, 4096), (2, 136)])
@pytest.mark.parametrize("with_r", [False, True])
def test_rmsnorm(M, H, with_r):
    x, r = f16(RNG.standard_normal((M, H))), f16(RNG.standard_normal((M, H)) * 3)
    w = inputs.norm_weight(H, seed=H)
    yref, href = dec.rmsnorm(x, w, 1e-6, r if with_r else None)
    xd, rd, wd = dev(x), dev(r), dev(w)
    y = _lib.laq_rmsnorm(xd, wd, 1e-6, R=rd if with_r else None, R_out=rd if with_r else None)
    close(host(y), yref, "y")
    if with_r:  # in place: R_out = R = fp16(x + r), at most one fp16 ulp from the exact sum
        assert np.allclose(host(rd).astype(np.float64), href.astype(np.float64), rtol=1e-3,
                           atol=1e-7)


def test_rmsnorm_rejects_bad_shapes():
    x = torch.zeros((1, 20), dtype=torch.float16, device=DEV)
    with pytest.raises(laq.LaqError) as e:
        _lib.laq_rmsnorm(x, torch.zeros(20, dtype=torch.float16, device=DEV), 1e-6)
    assert e.value.status == 4


# ---- q/k norm + rope + cache append ----

@pytest.mark.parametrize("pos", [[0], [5, 1000], [1023, 17, 300]])
def test_qk_norm_rope(pos):
    M, Hq, Hkv, D, L = len(pos), 32, 8, 128, 1024
    qkv = f16(RNG.standard_normal((M, (Hq + 2 * Hkv) * D)) * 2)
    qw, kw = inputs.norm_weight(D, 1), inputs.norm_weight(D, 2)
    kc0 = inputs.kv_cache(M, Hkv, L, D, seed=3)
    vc0 = inputs.kv_cache(M, Hkv, L, D, seed=4)
    kc, vc = dev(kc0), dev(vc0)
    q = _lib.laq_qk_norm_rope(dev(qkv), dev(qw), dev(kw), dev(np.array(pos, np.int32)), Hq,
                              Hkv, 1e6, 1e-6, kc, vc)
    qr, kr, vr = dec.qk_norm_rope(qkv, qw, kw, pos, Hq, Hkv, 1e6, 1e-6, D)
    close(host(q), qr, "q")
    kh, vh = host(kc), host(vc)
    for m, p in enumerate(pos):
        close(kh[m, :, p], kr[m], "k")
        assert np.array_equal(vh[m, :, p], vr[m])
        mask = np.ones(L, bool)
        mask[p] = False
        assert np.array_equal(kh[m][:, mask], kc0[m][:, mask])
        assert np.array_equal(vh[m][:, mask], vc0[m][:, mask])


def test_qk_norm_rope_position_outside_the_cache_stores_nothing():
    M, Hq, Hkv, D, L = 2, 4, 2, 128, 16
    qkv = f16(RNG.standard_normal((M, (Hq + 2 * Hkv) * D)))
    qw, kw = inputs.norm_weight(D, 5), inputs.norm_weight(D, 6)
    kc0, vc0 = inputs.kv_cache(M, Hkv, L, D, 7), inputs.kv_cache(M, Hkv, L, D, 8)
    kc, vc = dev(kc0), dev(vc0)
    pos = [L, -1]
    q = _lib.laq_qk_norm_rope(dev(qkv), dev(qw), dev(kw), dev(np.array(pos, np.int32)), Hq,
                              Hkv, 1e6, 1e-6, kc, vc)
    qr, _, _ = dec.qk_norm_rope(qkv, qw, kw, pos, Hq, Hkv, 1e6, 1e-6, D)
    close(host(q), qr, "q")
    assert np.array_equal(host(kc), kc0) and np.array_equal(host(vc), vc0)


# ---- attention ----

@pytest.mark.parametrize("lens", [[1], [63], [64], [65], [200, 7], [256, 129, 1]])
def test_attention(lens):
    M, Hq, Hkv, D, L = len(lens), 32, 8, 128, 256
    q = f16(RNG.standard_normal((M, Hq, D)))
    kc, vc = inputs.kv_cache(M, Hkv, L, D, 11), inputs.kv_cache(M, Hkv, L, D, 12)
    ws = _lib.attention_workspace(M, Hq, L, DEV)
    out = _lib.laq_attention_decode(dev(q), dev(kc), dev(vc), dev(np.array(lens, np.int32)),
                                    1 / math.sqrt(D), ws)
    close(host(out), dec.attention(q, kc, vc, lens, 1 / math.sqrt(D)), "attention")


def test_attention_empty_and_clamped_lengths():
    M, Hq, Hkv, D, L = 3, 8, 2, 128, 70
    q = f16(RNG.standard_normal((M, Hq, D)))
    kc, vc = inputs.kv_cache(M, Hkv, L, D, 13), inputs.kv_cache(M, Hkv, L, D, 14)
    lens = np.array([0, L + 50, -3], np.int32)
    ws = _lib.attention_workspace(M, Hq, L, DEV)
    out = host(_lib.laq_attention_decode(dev(q), dev(kc), dev(vc), dev(lens), 0.1, ws))
    ref = dec.attention(q, kc, vc, lens, 0.1)
    assert not out[0].any() and not out[2].any()
    close(out[1], ref[1], "clamped")


def test_attention_workspace_too_small():
    q = torch.zeros((1, 8, 128), dtype=torch.float16, device=DEV)
    kv = torch.zeros((1, 2, 64, 128), dtype=torch.float16, device=DEV)
    ws = torch.zeros((4,), dtype=torch.float32, device=DEV)
    with pytest.raises(laq.LaqError) as e:
        _lib.laq_attention_decode(q, kv, kv, torch.ones(1, dtype=torch.int32, device=DEV), 0.1, ws)
    assert e.value.status == 10


# ---- attention with the q/k norm, rotation and cache append folded in ----

def oracle_attention_qkv(qkv, qw, kw, pos, Hq, Hkv, kc0, vc0, scale):
    q, k, v = dec.qk_norm_rope(qkv, qw, kw, pos, Hq, Hkv, 1e6, 1e-6, 128)
    kc, vc = kc0.copy(), vc0.copy()
    L = kc.shape[2]
    for m, p in enumerate(pos):
        if 0 <= p < L:
            kc[m, :, p], vc[m, :, p] = k[m], v[m]
    lens = [min(max(p + 1, 0), L) for p in pos]
    return dec.attention(q, kc, vc, lens, scale), kc, vc


@pytest.mark.parametrize("pos", [[0], [63], [64], [100, 5], [255, 127, 191], [300], [-1, 70]])
def test_attention_qkv(pos):
    M, Hq, Hkv, D, L = len(pos), 32, 8, 128, 256
    qkv = f16(RNG.standard_normal((M, (Hq + 2 * Hkv) * D)) * 2)
    qw, kw = inputs.norm_weight(D, 21), inputs.norm_weight(D, 22)
    kc0, vc0 = inputs.kv_cache(M, Hkv, L, D, 23), inputs.kv_cache(M, Hkv, L, D, 24)
    scale = 1 / math.sqrt(D)
    ref, rk, rv = oracle_attention_qkv(qkv, qw, kw, pos, Hq, Hkv, kc0, vc0, scale)
    kc, vc = dev(kc0), dev(vc0)
    ws = _lib.attention_qkv_workspace(M, Hq, Hkv, L, DEV)
    args = (dev(qkv), dev(qw), dev(kw), dev(np.array(pos, np.int32)), Hq, Hkv, 1e6, 1e-6, kc, vc,
            scale, ws)
    out1 = host(_lib.laq_attention_qkv(*args))
    out2 = host(_lib.laq_attention_qkv(*args))   # a repeated call agrees bit for bit
    close(out1, ref, "attention_qkv")
    assert np.array_equal(out1, out2)
    close(host(kc), rk, "k cache")
    kh, vh = host(kc), host(vc)
    for m, p in enumerate(pos):
        if not 0 <= p < L:
            assert np.array_equal(kh[m], kc0[m]) and np.array_equal(vh[m], vc0[m])
        if p < 0:
            assert not out1[m].any()


# ---- SiLU * up, embedding, argmax ----

@pytest.mark.parametrize("M,I", [(1, 9728), (4, 24)])
def test_silu_mul(M, I):
    gu = f16(RNG.standard_normal((M, 2 * I)) * 4)
    close(host(_lib.laq_silu_mul(dev(gu))), dec.silu_mul(gu), "silu")


def test_embed_and_argmax():
    V, H = 1000, 2560
    E = inputs.embedding(V, H, seed=1)
    toks = np.array([0, 999, 1000, -5, 123], np.int32)
    X = host(_lib.laq_embed(dev(E), dev(toks)))
    assert np.array_equal(X, dec.embed(E, toks))
    logits = f16(RNG.standard_normal((4, 151936)))
    logits[1, 77] = logits[1, 99] = 50.0           # tie: the smaller index wins
    logits[2, :] = np.nan
    logits[2, 5000] = 1.0                          # NaN never wins
    logits[3, :] = -np.inf                         # no winner: 0
    logits[3, 7] = np.nan
    got = host(_lib.laq_argmax(dev(logits)))
    assert list(got) == list(dec.argmax(logits))
    assert got[1] == 77 and got[2] == 5000 and got[3] == 0
    # unaligned rows (V % 8 != 0) take the scalar path
    odd = f16(RNG.standard_normal((3, 1001)))
    odd[2, 1000] = 9.0
    assert list(host(_lib.laq_argmax(dev(odd)))) == list(dec.argmax(odd))


# ---- GEMV with the RMSNorm or SiLU*up prologue ----

def quantized(K, N, bits, seed):
    from oracle import c_oracle
    W = inputs.weights(K, N, seed=seed)
    codes, s, z = c_oracle.quantize_rtn(W, bits)
    packed = laq.laq_pack(dev(codes), bits)
    return (codes, s, z), (packed, dev(s), dev(z))


CFG = [None, laq.GemmConfig.make(2, 4, 8, 3, 1), laq.GemmConfig.make(1, 8, 1, 16, 0)]


@pytest.mark.parametrize("M", [1, 3, 16])
@pytest.mark.parametrize("ci", [0, 1, 2])
@pytest.mark.parametrize("with_r", [False, True])
def test_gemm_rmsnorm_prologue(M, ci, with_r):
    K, N, bits = 2560, 272, 3
    ref_q, (packed, s, z) = quantized(K, N, bits, seed=40 + M)
    x = f16(RNG.standard_normal((M, K)))
    r = f16(RNG.standard_normal((M, K)) * 2)
    w = inputs.norm_weight(K, seed=5)
    y_in, h = dec.rmsnorm(x, w, 1e-6, r if with_r else None)
    ref = dec.linear(y_in, ref_q)
    rd = dev(r)
    r_out = torch.zeros((M, K), dtype=torch.float16, device=DEV)
    Y = _lib.laq_gemm_wxg128_prologue(dev(x), packed, s, z, bits, _lib.PROLOGUE_RMSNORM,
                                      R=rd if with_r else None, R_out=r_out, w=dev(w), eps=1e-6,
                                      config=CFG[ci])
    close(host(Y), ref, "rmsnorm prologue")
    assert np.allclose(host(r_out).astype(np.float64), h.astype(np.float64), rtol=1e-3, atol=1e-7)


@pytest.mark.parametrize("M", [1, 4])
@pytest.mark.parametrize("ci", [0, 1])
def test_gemm_silu_prologue(M, ci):
    I, N, bits = 1280, 80, 4
    ref_q, (packed, s, z) = quantized(I, N, bits, seed=60 + M)
    gu = f16(RNG.standard_normal((M, 2 * I)) * 3)
    # gates at the ends of the range: silu -> -0 (e^-g overflows) and silu(g) = g
    gu[:, :8] = f16([-65504.0, -100.0, -88.0, -87.0, 60.0, 11.0, 0.0, -0.0])
    ref = dec.linear(dec.silu_mul(gu), ref_q)
    Y = _lib.laq_gemm_wxg128_prologue(dev(gu), packed, s, z, bits, _lib.PROLOGUE_SILU_MUL,
                                      config=CFG[ci])
    close(host(Y), ref, "silu prologue")


def test_gemm_prologue_rejects_aliasing():
    _, (packed, s, z) = quantized(256, 32, 3, seed=1)
    x = torch.zeros((1, 256), dtype=torch.float16, device=DEV)
    r = torch.zeros((1, 256), dtype=torch.float16, device=DEV)
    w = torch.ones(256, dtype=torch.float16, device=DEV)
    with pytest.raises(laq.LaqError) as e:
        _lib.laq_gemm_wxg128_prologue(x, packed, s, z, 3, _lib.PROLOGUE_RMSNORM, R=r, R_out=r, w=w)
    assert e.value.status == 4


# ---- one whole decode step (2 layers, real Qwen3-4B widths, small vocabulary) ----

def oracle_model(st):
    """The decode step ``st`` (a DecodeStep) as numpy arrays for oracle.decoder.decode_step: the
    quantized projections as (codes, s, z) re-derived on the host by the C oracle from the same
    fp16 weights, the norm weights, the rotation tables and the embedding."""
    from oracle import c_oracle
    layers = []
    for l in range(st.layers):
        ws = []
        for _, members, _, _ in st.wp.linears[4 * l:4 * l + 4]:
            W = st.wp.weight(l, members).cpu().numpy()
            ws.append(c_oracle.quantize_rtn(W, st.bits))
        nw = {k: v.cpu().numpy() for k, v in st.norms[l].items()}
        layers.append(dict(qkv=ws[0], o=ws[1], gate_up=ws[2], down=ws[3], **nw))
        if st.rot:
            layers[-1]["rot"] = {name: (t["alpha"].cpu().numpy(), t["pairs"].cpu().numpy(),
                                        t["theta"].cpu().numpy())
                                 for name, t in st.rot[l].items()}
    E = st.E.cpu().numpy()
    return {"E": E, "layers": layers, "final_w": st.final_w.cpu().numpy(),
            "lm": c_oracle.quantize_rtn(E.T.copy(), st.bits), "Hq": st.Hq, "Hkv": st.Hkv,
            "D": st.D, "I": st.I, "theta": st.theta, "eps": st.eps}


@pytest.mark.parametrize("bits,M,fused,norms,rot", [
    (3, 1, True, True, 0), (4, 2, True, True, 0), (3, 2, False, False, 0), (4, 1, True, False, 0),
    # the rotation-based variant: a pairwise rotation before every projection of a layer
    (3, 1, True, True, 4), (4, 2, False, False, 2)])
def test_decode_step(bits, M, fused, norms, rot):
    from paper_2605_08755_gb300.decode_step import DecodeStep
    st = DecodeStep(bits=bits, M=M, layers=2, context=96, vocab=4096, seed=3,
                    fused_attention=fused, fused_norms=norms, rotation_rounds=rot)
    kc0 = [host(c).copy() for c in st.kc]
    vc0 = [host(c).copy() for c in st.vc]
    tokens = host(st.tokens)
    pos = [st.context - 1] * M
    st.run()
    logits, nxt = host(st.logits), host(st.next)
    model = oracle_model(st)
    rl, rn, rk, rv = dec.decode_step(model, tokens, pos, kc0, vc0)
    close(logits, rl, "logits")
    # the greedy token: equal unless the oracle's top two logits are within the tolerance
    tol = 5e-3 * np.abs(rl.astype(np.float64)).max() + 1e-3
    for m in range(M):
        top = np.sort(rl[m].astype(np.float64))[-2:]
        if top[1] - top[0] > 2 * tol:
            assert nxt[m] == rn[m]
        assert nxt[m] == int(np.argmax(logits[m]))
    for l in range(2):
        close(host(st.kc[l])[:, :, pos[0]], rk[l][:, :, pos[0]], "k cache")
        close(host(st.vc[l])[:, :, pos[0]], rv[l][:, :, pos[0]], "v cache")
    # a CUDA-graph replay gives the same step
    g = st.capture()
    g.replay()
    assert np.array_equal(host(st.logits), logits)
