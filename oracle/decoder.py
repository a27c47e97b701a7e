"""CPU oracle for the decoder operations of one decode step (numpy, float64).

TEST INFRASTRUCTURE ONLY (like the rest of ``oracle``): the tests, ``smoke()`` and the
benchmark's CPU leg may use it; the product path never does.  It shares no code with the CUDA
library.

The paper measures decoding speed of quantized Qwen3 models (Sec. 5.2) but defines none of the
operations around the projections; each function below writes out the standard definition it
names, in float64, taking fp16 tensors and returning fp16 (rounded once), which are the points
where the CUDA path stores fp16:

* ``rmsnorm``        -- RMSNorm (root-mean-square layer normalisation with a weight) after the
                        residual add, h = fp16(x + r);
* ``qk_norm_rope``   -- per-head RMSNorm of q and k and the rotary position embedding in its
                        rotate-half form, angle p * theta^(-2i/D) for the pair (i, i + D/2);
* ``attention``      -- softmax attention of one query per head over the cached keys and values,
                        grouped-query heads (q head h reads kv head h // (Hq / Hkv));
* ``silu_mul``       -- SiLU(gate) * up, SiLU(x) = x / (1 + e^-x);
* ``embed`` / ``argmax`` -- row gather; the first index of the maximum;
* ``decode_step``    -- one token of a Qwen3-style decoder built from the above and the
                        quantized projections (Eq. (1), dequantized by the C oracle),
                        optionally with the online pairwise rotation of ``oracle.rotation`` on
                        the input of every projection of a layer.
"""
import math

import numpy as np

from . import c_oracle
from . import rotation


def _f64(a):
    return np.asarray(a, np.float16).astype(np.float64)


def _f16(a):
    return np.asarray(a, np.float64).astype(np.float16)


def rmsnorm(x, w, eps, r=None):
    """Rows of x [M, H]: h = fp16(x + r) (h = x without r); y = h / sqrt(mean(h^2) + eps) * w.
    Returns (y, h) in fp16."""
    h = _f64(x) if r is None else _f64(_f16(_f64(x) + _f64(r)))
    ms = np.mean(h * h, axis=1, keepdims=True)
    y = h / np.sqrt(ms + eps) * _f64(w)[None, :]
    return _f16(y), _f16(h)


def rope(x, p, theta):
    """Rotate-half rotary embedding of the head vectors x [..., D] at position p (float64 in,
    float64 out): for i < D/2, a_i = p * theta^(-2i / D),
    (x_i, x_{i+D/2}) -> (x_i cos a_i - x_{i+D/2} sin a_i, x_{i+D/2} cos a_i + x_i sin a_i)."""
    x = np.asarray(x, np.float64)
    D = x.shape[-1]
    half = D // 2
    i = np.arange(half, dtype=np.float64)
    a = float(p) * theta ** (-2.0 * i / D)
    c, s = np.cos(a), np.sin(a)
    x1, x2 = x[..., :half], x[..., half:]
    return np.concatenate([x1 * c - x2 * s, x2 * c + x1 * s], axis=-1)


def qk_norm_rope(qkv, q_w, k_w, pos, Hq, Hkv, theta, eps, D=128):
    """qkv [M, (Hq + 2 Hkv) D] -> (q [M, Hq, D], k [M, Hkv, D], v [M, Hkv, D]) in fp16:
    q and k heads RMS-normalised with their weights, then rotated at pos[m]; v unchanged."""
    qkv = _f64(qkv)
    M = qkv.shape[0]
    heads = qkv.reshape(M, Hq + 2 * Hkv, D)
    q, k, v = heads[:, :Hq], heads[:, Hq:Hq + Hkv], heads[:, Hq + Hkv:]

    def norm(x, w):
        return x / np.sqrt(np.mean(x * x, axis=-1, keepdims=True) + eps) * _f64(w)

    qo = np.stack([rope(norm(q[m], q_w), pos[m], theta) for m in range(M)])
    ko = np.stack([rope(norm(k[m], k_w), pos[m], theta) for m in range(M)])
    return _f16(qo), _f16(ko), _f16(v)


def attention(q, k_cache, v_cache, lens, scale):
    """q [M, Hq, D]; caches [M, Hkv, L, D]; row m attends to its first lens[m] tokens:
    out[m, h] = sum_t softmax_t(scale * q[m, h] . k[m, g, t]) v[m, g, t], g = h // (Hq / Hkv).
    Rows with no token give zeros.  fp16 out."""
    q, K, V = _f64(q), _f64(k_cache), _f64(v_cache)
    M, Hq, D = q.shape
    Hkv = K.shape[1]
    G = Hq // Hkv
    out = np.zeros((M, Hq, D))
    for m in range(M):
        n = int(min(max(int(lens[m]), 0), K.shape[2]))
        if n == 0:
            continue
        for h in range(Hq):
            g = h // G
            s = scale * (K[m, g, :n] @ q[m, h])
            e = np.exp(s - s.max())
            out[m, h] = (e / e.sum()) @ V[m, g, :n]
    return _f16(out)


def silu_mul(gate_up):
    """[M, 2I] -> [M, I]: silu(g) * u with g the first I columns, u the last I."""
    gu = _f64(gate_up)
    I = gu.shape[1] // 2
    g, u = gu[:, :I], gu[:, I:]
    with np.errstate(over="ignore"):  # g << 0: e^-g = inf and g / inf = -0, silu's limit
        return _f16(g / (1.0 + np.exp(-g)) * u)


def embed(E, tokens):
    E = np.asarray(E, np.float16)
    V, H = E.shape
    return np.stack([E[t] if 0 <= t < V else np.zeros(H, np.float16) for t in tokens])


def argmax(logits):
    """First index of the maximum of each row (NaN never wins; all-NaN or all -inf rows: 0)."""
    L = _f64(logits)
    out = []
    for row in L:
        best, bi = -math.inf, None
        for i, v in enumerate(row):
            if v > best:
                best, bi = v, i
        out.append(0 if bi is None else bi)
    return np.array(out, np.int32)


def linear(x, q):
    """fp16 x [M, K] times the dequantized weight of q = (codes, s, z) (Eq. (1)), fp16 out."""
    codes, s, z = q
    return _f16(_f64(x) @ c_oracle.dequant(codes, s, z))


def decode_step(model, tokens, pos, k_caches, v_caches):
    """One decode step of a Qwen3-style decoder for the rows' new tokens at positions pos.

    ``model``: dict with ``E`` [V, H] (embedding), ``layers`` (each a dict of quantized
    projections ``qkv``, ``o``, ``gate_up``, ``down`` as (codes, s, z) and fp16 norm weights
    ``in_w``, ``post_w``, ``q_w``, ``k_w``), ``final_w``, ``lm`` (quantized [H, V]) and the
    scalars ``Hq``, ``Hkv``, ``D``, ``I``, ``theta``, ``eps``.  A layer may carry ``rot``: per
    projection name a table (alpha, pairs, angles) of ``oracle.rotation`` applied to that
    projection's input (fp16 in, fp16 out) before it.  ``k_caches`` / ``v_caches``:
    per layer fp16 [M, Hkv, L, D]; the new token's k and v are written at pos[m] (copies are
    returned with them).  Returns (logits fp16 [M, V], next tokens, new caches)."""
    Hq, Hkv, D = model["Hq"], model["Hkv"], model["D"]
    theta, eps = model["theta"], model["eps"]
    scale = 1.0 / math.sqrt(D)
    kcs = [np.array(c, np.float16, copy=True) for c in k_caches]
    vcs = [np.array(c, np.float16, copy=True) for c in v_caches]
    x = embed(model["E"], tokens)
    r = x
    h, _ = rmsnorm(x, model["layers"][0]["in_w"], eps)
    lens = [p + 1 for p in pos]
    for li, Lw in enumerate(model["layers"]):
        rot = Lw.get("rot", {})

        def proj(name, x):
            if name in rot:
                alpha, pairs, angles = rot[name]
                x = rotation.pairwise_rotate(x, alpha, pairs, angles)
            return linear(x, Lw[name])

        if li > 0:
            h, r = rmsnorm(d, Lw["in_w"], eps, r)
        qkv = proj("qkv", h)
        q, k, v = qk_norm_rope(qkv, Lw["q_w"], Lw["k_w"], pos, Hq, Hkv, theta, eps, D)
        for m, p in enumerate(pos):
            kcs[li][m, :, p] = k[m]
            vcs[li][m, :, p] = v[m]
        a = attention(q, kcs[li], vcs[li], lens, scale).reshape(len(tokens), Hq * D)
        o = proj("o", a)
        h, r = rmsnorm(o, Lw["post_w"], eps, r)
        gu = proj("gate_up", h)
        d = proj("down", silu_mul(gu))
    h, _ = rmsnorm(d, model["final_w"], eps, r)
    logits = linear(h, model["lm"])
    return logits, argmax(logits), kcs, vcs
