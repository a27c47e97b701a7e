"""Pins of the decode-step oracle (oracle/decoder.py) against closed forms and invariants of the
definitions it restates -- RMSNorm, the rotate-half rotary embedding, softmax attention with
grouped kv heads, SiLU, argmax -- and one composed step whose answer follows by hand.  CPU only."""
import math

import numpy as np
import pytest

from oracle import c_oracle
from oracle import decoder as dec
from paper_2605_08755_gb300 import inputs

RNG = np.random.default_rng(1234)


def f16(a):
    return np.asarray(a, np.float64).astype(np.float16)


# ---- RMSNorm ----

@pytest.mark.parametrize("c", [0.5, -3.0, 1e-3])
def test_rmsnorm_constant_row(c):
    H, eps = 64, 1e-6
    w = f16(RNG.uniform(0.5, 1.5, H))
    y, h = dec.rmsnorm(f16(np.full((1, H), c)), w, eps)
    c16 = float(np.float16(c))
    expect = c16 / math.sqrt(c16 * c16 + eps) * w.astype(np.float64)
    assert np.array_equal(h[0], f16(np.full(H, c16)))
    assert np.array_equal(y[0], f16(expect))


def test_rmsnorm_unit_mean_square_and_residual():
    H = 2560
    x, r = f16(RNG.standard_normal((3, H))), f16(RNG.standard_normal((3, H)))
    y, h = dec.rmsnorm(x, f16(np.ones(H)), 0.0, r)
    # h is the fp16 sum; with w = 1, eps = 0 the output rows have mean square 1 (to fp16)
    assert np.array_equal(h, f16(x.astype(np.float64) + r.astype(np.float64)))
    ms = np.mean(y.astype(np.float64) ** 2, axis=1)
    assert np.all(np.abs(ms - 1.0) < 2e-3)


# ---- rotary embedding ----

def test_rope_position_zero_is_identity_and_pairs_keep_their_norm():
    x = RNG.standard_normal((5, 128))
    assert np.array_equal(dec.rope(x, 0, 1e6), x)
    y = dec.rope(x, 37, 1e6)
    n0 = x[:, :64] ** 2 + x[:, 64:] ** 2
    n1 = y[:, :64] ** 2 + y[:, 64:] ** 2
    assert np.allclose(n0, n1, rtol=1e-12, atol=1e-12)


def test_rope_rotations_compose():
    x = RNG.standard_normal(128)
    a = dec.rope(dec.rope(x, 11, 1e4), 29, 1e4)
    b = dec.rope(x, 40, 1e4)
    assert np.allclose(a, b, rtol=0, atol=1e-12)


def test_rope_hand_example():
    # D = 4, theta = 100: pair 0 turns by p, pair 1 by p / 10
    x = np.array([1.0, 2.0, 3.0, 4.0])
    p = 2
    a0, a1 = 2.0, 0.2
    expect = [1 * math.cos(a0) - 3 * math.sin(a0), 2 * math.cos(a1) - 4 * math.sin(a1),
              3 * math.cos(a0) + 1 * math.sin(a0), 4 * math.cos(a1) + 2 * math.sin(a1)]
    assert np.allclose(dec.rope(x, p, 100.0), expect, rtol=0, atol=1e-15)


def test_qk_norm_rope_leaves_v_and_normalises_at_position_zero():
    Hq, Hkv, D = 4, 2, 128
    qkv = f16(RNG.standard_normal((2, (Hq + 2 * Hkv) * D)))
    qw, kw = f16(RNG.uniform(0.5, 1.5, D)), f16(RNG.uniform(0.5, 1.5, D))
    q, k, v = dec.qk_norm_rope(qkv, qw, kw, [0, 0], Hq, Hkv, 1e6, 1e-6, D)
    heads = qkv.reshape(2, Hq + 2 * Hkv, D)
    assert np.array_equal(v, heads[:, Hq + Hkv:])
    for m in range(2):
        for h in range(Hq):
            y, _ = dec.rmsnorm(heads[m, h][None], qw, 1e-6)
            assert np.array_equal(q[m, h], y[0])


# ---- attention ----

def test_attention_single_token_returns_its_value():
    q = f16(RNG.standard_normal((1, 4, 128)))
    K = f16(RNG.standard_normal((1, 2, 8, 128)))
    V = f16(RNG.standard_normal((1, 2, 8, 128)))
    out = dec.attention(q, K, V, [1], 0.1)
    for h in range(4):
        assert np.array_equal(out[0, h], V[0, h // 2, 0])


def test_attention_uniform_scores_average_the_values():
    q = f16(np.zeros((1, 2, 128)))
    V = f16(RNG.standard_normal((1, 1, 10, 128)))
    out = dec.attention(q, f16(RNG.standard_normal((1, 1, 10, 128))), V, [7], 0.5)
    assert np.array_equal(out[0, 0], f16(V[0, 0, :7].astype(np.float64).mean(axis=0)))


def test_attention_large_scale_picks_the_aligned_key_per_group():
    # kv head g holds keys e_j; q head h points at key 3 + g with a huge scale; GQA: heads
    # 2g and 2g + 1 read kv head g
    Hq, Hkv, L, D = 4, 2, 6, 128
    K = np.zeros((1, Hkv, L, D))
    for g in range(Hkv):
        for t in range(L):
            K[0, g, t, t] = 1.0
    V = f16(RNG.standard_normal((1, Hkv, L, D)))
    q = np.zeros((1, Hq, D))
    for h in range(Hq):
        q[0, h, 3 + h // 2] = 1.0
    out = dec.attention(f16(q), f16(K), V, [L], 200.0)
    for h in range(Hq):
        assert np.array_equal(out[0, h], V[0, h // 2, 3 + h // 2])


def test_attention_empty_row_is_zero():
    out = dec.attention(f16(np.ones((1, 1, 128))), f16(np.ones((1, 1, 4, 128))),
                        f16(np.ones((1, 1, 4, 128))), [0], 1.0)
    assert not out.any()


# ---- SiLU * up, embedding, argmax ----

def test_silu_mul_closed_forms():
    gu = f16([[0.0, 1.0, -1.0, 2.0, 2.0, 3.0]])  # g = (0, 1, -1), u = (2, 2, 3)
    y = dec.silu_mul(gu)[0].astype(np.float64)
    expect = [0.0, 2.0 / (1.0 + math.exp(-1.0)), -3.0 / (1.0 + math.exp(1.0))]
    assert np.array_equal(dec.silu_mul(gu)[0], f16(expect))
    assert y[0] == 0.0


def test_embed_and_argmax():
    E = f16(RNG.standard_normal((10, 16)))
    X = dec.embed(E, [3, -1, 10])
    assert np.array_equal(X[0], E[3]) and not X[1].any() and not X[2].any()
    logits = f16([[1.0, 5.0, 5.0, -2.0], [np.nan, 0.5, np.nan, 0.5], [-np.inf] * 4])
    assert list(dec.argmax(logits)) == [1, 1, 0]


# ---- one composed step with a closed-form answer ----

def zero_weight(K, N, bits=3):
    # codes equal to the zero point dequantize to exactly 0 (Eq. (1))
    codes = np.full((K, N), 2, np.uint8)
    s = np.full((K // 128, N), np.float16(0.01))
    z = np.full((K // 128, N), 2, np.uint8)
    return codes, s, z


def test_decode_step_with_zero_attention_and_mlp_outputs():
    # o and down dequantize to 0, so the residual stream stays the embedding and the logits
    # are rmsnorm(E[t]) * final_w times the LM head; the caches get the new k, v at pos.
    H, Hq, Hkv, D, I, V, L = 256, 2, 1, 128, 256, 32, 8
    eps, theta = 1e-6, 1e6
    E = f16(RNG.standard_normal((V, H)))
    lmW = f16(RNG.standard_normal((H, V)) * 0.05)
    lm = c_oracle.quantize_rtn(lmW, 4)
    qkvW = f16(RNG.standard_normal((H, (Hq + 2 * Hkv) * D)) * 0.05)
    guW = f16(RNG.standard_normal((H, 2 * I)) * 0.05)
    layer = {"qkv": c_oracle.quantize_rtn(qkvW, 3), "o": zero_weight(Hq * D, H),
             "gate_up": c_oracle.quantize_rtn(guW, 3), "down": zero_weight(I, H),
             "in_w": f16(np.ones(H)), "post_w": f16(np.ones(H)),
             "q_w": f16(np.ones(D)), "k_w": f16(np.ones(D))}
    final_w = f16(RNG.uniform(0.5, 1.5, H))
    model = {"E": E, "layers": [layer, layer], "final_w": final_w, "lm": lm, "Hq": Hq,
             "Hkv": Hkv, "D": D, "I": I, "theta": theta, "eps": eps}
    kc = [f16(RNG.standard_normal((2, Hkv, L, D))) for _ in range(2)]
    vc = [f16(RNG.standard_normal((2, Hkv, L, D))) for _ in range(2)]
    tokens, pos = [5, 17], [3, 6]
    logits, nxt, kcs, vcs = dec.decode_step(model, tokens, pos, kc, vc)
    x = E[tokens]
    h, _ = dec.rmsnorm(x, final_w, eps)   # r + 0 + 0 == r exactly
    expect = f16(h.astype(np.float64) @ c_oracle.dequant(*lm))
    assert np.array_equal(logits, expect)
    assert list(nxt) == list(dec.argmax(expect))
    # caches: only the new positions changed; there, v is the raw v projection of h_in
    h_in, _ = dec.rmsnorm(x, layer["in_w"], eps)
    qkv = dec.linear(h_in, layer["qkv"])
    _, k_new, v_new = dec.qk_norm_rope(qkv, layer["q_w"], layer["k_w"], pos, Hq, Hkv, theta,
                                       eps, D)
    for m, p in enumerate(pos):
        mask = np.ones(L, bool)
        mask[p] = False
        assert np.array_equal(kcs[0][m][:, mask], kc[0][m][:, mask])
        assert np.array_equal(vcs[0][m, :, p], v_new[m])
        assert np.array_equal(kcs[0][m, :, p], k_new[m])


def test_decode_step_with_identity_rotations_is_unchanged():
    # zero angles and unit scales: the rotated step equals the plain one bit for bit; one real
    # rotation on the o input changes the logits
    H, Hq, Hkv, D, I, V, L = 256, 2, 1, 128, 256, 32, 8
    E = f16(RNG.standard_normal((V, H)))
    q = lambda K, N: c_oracle.quantize_rtn(f16(RNG.standard_normal((K, N)) * 0.05), 3)
    layer = {"qkv": q(H, (Hq + 2 * Hkv) * D), "o": q(Hq * D, H), "gate_up": q(H, 2 * I),
             "down": q(I, H), "in_w": f16(np.ones(H)), "post_w": f16(np.ones(H)),
             "q_w": f16(np.ones(D)), "k_w": f16(np.ones(D))}
    model = {"E": E, "layers": [layer], "final_w": f16(np.ones(H)), "lm": q(H, V), "Hq": Hq,
             "Hkv": Hkv, "D": D, "I": I, "theta": 1e6, "eps": 1e-6}
    kc = [f16(RNG.standard_normal((1, Hkv, L, D)))]
    vc = [f16(RNG.standard_normal((1, Hkv, L, D)))]
    plain = dec.decode_step(model, [3], [4], kc, vc)[0]
    ident = {}
    for name, K in (("qkv", H), ("o", Hq * D), ("gate_up", H), ("down", I)):
        pairs = inputs.rotation(K, 2, seed=K)[0]
        ident[name] = (f16(np.ones(K)), pairs, np.zeros((K // 128, 2, 64), np.float32))
    rotated = dec.decode_step({**model, "layers": [{**layer, "rot": ident}]}, [3], [4], kc, vc)[0]
    assert np.array_equal(rotated, plain)
    real = dict(ident)
    real["o"] = inputs.rotation(Hq * D, 2, seed=9)
    real["o"] = (real["o"][2], real["o"][0], real["o"][1])
    moved = dec.decode_step({**model, "layers": [{**layer, "rot": real}]}, [3], [4], kc, vc)[0]
    assert not np.array_equal(moved, plain)
