"""Pins of the CPU oracle to what Eq. (1) and plain mathematics fix (no GPU needed).

Every check here ties the oracle to something other than itself: a closed form (planted codes),
hand-computed fixtures (ties, single-code packing), invariants that Eq. (1) implies under the
documented readings, special cases that reduce to a library routine (numpy's binary16 decoder,
numpy.matmul), exact rational brute force on tiny inputs, and an independent numpy restatement.
"""
import os
from fractions import Fraction

import numpy as np
import pytest

from oracle import c_oracle as co
from oracle import ref_numpy as rn
from paper_2605_08755_gb300 import inputs
from tests.conftest import GOLDEN

pytestmark = pytest.mark.filterwarnings("ignore::RuntimeWarning")


def _planted(bits, G, N, seed, m, e):
    """W = s0 * (Q - z0) with s0 = m * 2^-e (m < 128, so every s0 * j, |j| <= 15, is exact in
    fp16), z0 per column, and codes 0 and 2^b - 1 present in every (group, column)."""
    rng = np.random.default_rng(seed)
    qmax = (1 << bits) - 1
    K = G * 128
    Q = rng.integers(0, qmax + 1, size=(K, N)).astype(np.int64)
    for g in range(G):
        Q[g * 128, :] = 0
        Q[g * 128 + 1 + (g % 5), :] = qmax
    z0 = rng.integers(0, qmax + 1, size=(G, N)).astype(np.int64)
    s0 = m * 2.0 ** -e
    Wf = s0 * (Q - np.repeat(z0, 128, axis=0))
    W = Wf.astype(np.float16)
    assert np.array_equal(W.astype(np.float64), Wf), "planted weights must be exact in fp16"
    return W, Q.astype(np.uint8), np.float16(s0), z0.astype(np.uint8)


@pytest.mark.parametrize("bits", [3, 4])
@pytest.mark.parametrize("m,e", [(1, 6), (3, 9), (127, 14), (5, 2), (1, 0)])
@pytest.mark.parametrize("impl", ["c", "numpy"])
def test_planted_codes_recovered_exactly(bits, m, e, impl):
    W, Q, s0, z0 = _planted(bits, G=3, N=24, seed=bits * 100 + m + e, m=m, e=e)
    q = (co if impl == "c" else rn).quantize_rtn(W, bits)
    codes, s, z = q
    assert np.all(s == s0)
    assert np.array_equal(z, z0)
    assert np.array_equal(codes, Q)


def _load_ties():
    blocks = []
    with open(os.path.join(GOLDEN, "eq1_ties.txt")) as f:
        for line in f:
            line = line.split("#")[0].split()
            if not line:
                continue
            if line[0] == "group":
                blocks.append({"bits": int(line[1]), "s": int(line[2]) / 128.0,
                               "z": int(line[3]), "w": []})
            else:
                blocks[-1]["w"].append((int(line[1]) / 128.0, int(line[2])))
    return blocks


@pytest.mark.parametrize("impl", ["c", "numpy"])
def test_eq1_ties_round_half_even_before_adding_z(impl):
    for blk in _load_ties():
        col = np.zeros(128, np.float64)
        for i, (w, _) in enumerate(blk["w"]):
            col[i] = w
        W = col.astype(np.float16).reshape(128, 1)
        codes, s, z = (co if impl == "c" else rn).quantize_rtn(W, blk["bits"])
        assert float(s[0, 0]) == blk["s"]
        assert int(z[0, 0]) == blk["z"]
        for i, (_, q) in enumerate(blk["w"]):
            assert int(codes[i, 0]) == q, (blk["bits"], i)
        assert np.all(codes[len(blk["w"]):, 0] == blk["z"])


def test_ties_fixture_rejects_round_after_adding_z():
    """A planted mistake in a copy of the numpy oracle (round(w/s + z) instead of
    round(w/s) + z) must fail the tie fixture."""
    for blk in _load_ties():
        wrong = [int(np.clip(np.rint(w / blk["s"] + blk["z"]), 0, (1 << blk["bits"]) - 1))
                 for w, _ in blk["w"]]
        right = [q for _, q in blk["w"]]
        assert wrong != right


@pytest.mark.parametrize("c", [0.013, -0.013, 0.0, -0.0, 65504.0, -65504.0, 2.0 ** -20,
                               -(2.0 ** -24), 1.0, -3.5])
@pytest.mark.parametrize("bits", [3, 4])
@pytest.mark.parametrize("impl", ["c", "numpy"])
def test_constant_groups_are_exact(c, bits, impl):
    W = np.full((256, 3), c, np.float16)
    W[128:, 1] = np.float16(0.5)  # a second group with another constant
    codes, s, z = (co if impl == "c" else rn).quantize_rtn(W, bits)
    What = co.dequant(codes, s, z)
    assert np.array_equal(What, W.astype(np.float64))


@pytest.mark.parametrize("bits", [3, 4])
@pytest.mark.parametrize("outliers", [False, True])
def test_invariants_code_range_and_half_step_error(bits, outliers):
    qmax = (1 << bits) - 1
    W = inputs.weights(512, 96, seed=11 + bits, outliers=outliers)
    W[:128, 5] = np.abs(W[:128, 5])           # an all-non-negative group
    W[128:256, 7] = -np.abs(W[128:256, 7])    # an all-non-positive group
    W[256:384, 9] = np.float16(2.0 ** -24) * np.arange(128).astype(np.float16)  # tiny range
    codes, s, z = co.quantize_rtn(W, bits)
    assert codes.max() <= qmax and z.max() <= qmax
    sv = s.astype(np.float64)
    What = co.dequant(codes, s, z)
    err = np.abs(What - W.astype(np.float64))
    bound = np.repeat(sv, 128, axis=0) / 2
    assert np.all(err <= bound)


def test_half_decoder_matches_numpy_binary16():
    bits = np.arange(0x10000, dtype=np.uint32).astype(np.uint16)
    ref = bits.view(np.float16).astype(np.float64)
    got = np.array([co.half_to_double(int(b)) for b in bits[::7]])
    r = ref[::7]
    same = (got == r) | (np.isnan(got) & np.isnan(r))
    assert np.all(same)


@pytest.mark.parametrize("bits", [3, 4])
@pytest.mark.parametrize("outliers", [False, True])
def test_c_oracle_matches_numpy_restatement(bits, outliers):
    W = inputs.weights(1024, 128, seed=5, outliers=outliers)
    c1 = co.quantize_rtn(W, bits)
    c2 = rn.quantize_rtn(W, bits)
    for a, b in zip(c1, c2):
        assert np.array_equal(np.asarray(a).view(np.uint8), np.asarray(b).view(np.uint8))
    X = inputs.activations(3, 1024, seed=5)
    y1 = co.gemm(X, *c1)
    y2 = rn.gemm(X, *c2)
    assert np.allclose(y1, y2, rtol=1e-12, atol=1e-12)


# ---------------- packing ----------------

@pytest.mark.parametrize("bits", [3, 4])
def test_layout_is_a_bijection(bits):
    wpl = 8 if bits == 4 else 6
    seen = set()
    for l in range(32):
        for w in range(wpl):
            for b in range(32):
                seen.add(co.layout_bit(bits, l, w, b))
    assert len(seen) == 32 * wpl * 32 == 128 * 16 * bits
    assert all(0 <= kk < 128 and 0 <= nn < 16 and 0 <= cb < bits for kk, nn, cb in seen)
    offs = {co.word_offset(bits, l, w) for l in range(32) for w in range(wpl)}
    assert offs == set(range(32 * wpl))


def _load_single_codes():
    rows = []
    with open(os.path.join(GOLDEN, "pack_single_codes.txt")) as f:
        for line in f:
            line = line.split("#")[0].split()
            if not line:
                continue
            bits, k, n, code = (int(v) for v in line[:4])
            words = {int(o): int(v, 16) for o, v in (t.split(":") for t in line[4:])}
            rows.append((bits, k, n, code, words))
    return rows


@pytest.mark.parametrize("impl", ["c", "numpy"])
def test_pack_single_code_golden(impl):
    for bits, k, n, code, words in _load_single_codes():
        codes = np.zeros((128, 16), np.uint8)
        codes[k, n] = code
        packed = (co if impl == "c" else rn).pack(codes, bits)
        nz = {int(i): int(packed[i]) for i in np.nonzero(packed)[0]}
        assert nz == words, (bits, k, n, code)


@pytest.mark.parametrize("bits", [3, 4])
def test_pack_roundtrip_and_cross_implementation(bits):
    qmax = (1 << bits) - 1
    rng = np.random.default_rng(3)
    K, N = 384, 48
    cases = [rng.integers(0, qmax + 1, size=(K, N)).astype(np.uint8),
             np.zeros((K, N), np.uint8), np.full((K, N), qmax, np.uint8)]
    walk = np.zeros((K, N), np.uint8)
    for i in range(K * N // 7):
        walk.flat[i * 7] = 1 << (i % bits)
    cases.append(walk)
    for codes in cases:
        p_c = co.pack(codes, bits)
        p_n = rn.pack(codes, bits)
        assert p_c.size * 32 == K * N * bits
        assert np.array_equal(p_c, p_n)
        assert np.array_equal(co.unpack(p_c, K, N, bits), codes)
        assert np.array_equal(rn.unpack(p_c, K, N, bits), codes)


# ---------------- Y = X * W_hat ----------------

@pytest.mark.parametrize("bits", [3, 4])
def test_one_hot_x_gives_dequantized_row(bits):
    W = inputs.weights(256, 32, seed=2)
    codes, s, z = co.quantize_rtn(W, bits)
    What = co.dequant(codes, s, z)
    for k in (0, 1, 127, 128, 200, 255):
        X = np.zeros((1, 256), np.float16)
        X[0, k] = 1.0
        Y = co.gemm(X, codes, s, z)
        assert np.array_equal(Y[0], What[k])
        # hand-expanded: s * (q - z) of row k
        g = k // 128
        hand = [float(s[g, n]) * (int(codes[k, n]) - int(z[g, n])) for n in range(32)]
        assert np.array_equal(Y[0], np.array(hand))


@pytest.mark.parametrize("bits", [3, 4])
def test_ones_over_a_group_sums_the_group(bits):
    W = inputs.weights(384, 16, seed=4)
    codes, s, z = co.quantize_rtn(W, bits)
    X = np.zeros((1, 384), np.float16)
    X[0, 128:256] = 1.0
    Y = co.gemm(X, codes, s, z)
    for n in range(16):
        tot = sum(Fraction(float(s[1, n])) * (int(codes[k, n]) - int(z[1, n]))
                  for k in range(128, 256))
        assert Y[0, n] == float(tot)


def test_small_integer_x_with_power_of_two_scales_is_exact():
    """X in small integers and s a power of two: every product and partial sum is exact, so Y
    equals the exact rational sum; the same inputs are used to demand bit-exact GPU output."""
    rng = np.random.default_rng(9)
    bits = 3
    W, Q, s0, z0 = _planted(bits, G=2, N=16, seed=9, m=1, e=5)
    X = rng.integers(-3, 4, size=(2, 256)).astype(np.float16)
    codes, s, z = co.quantize_rtn(W, bits)
    Y = co.gemm(X, codes, s, z)
    for m in range(2):
        for n in range(16):
            exact = sum(Fraction(int(X[m, k])) * Fraction(float(s[k // 128, n])) *
                        (int(codes[k, n]) - int(z[k // 128, n])) for k in range(256))
            assert Y[m, n] == float(exact)
    assert np.array_equal(Y.astype(np.float16).astype(np.float64), Y)  # exact in fp16 too


@pytest.mark.parametrize("bits", [3, 4])
@pytest.mark.parametrize("M,N", [(1, 1), (2, 5), (3, 8)])
def test_brute_force_tiny(bits, M, N):
    W = inputs.weights(128, N, seed=M * 10 + N)
    X = inputs.activations(M, 128, seed=M + N)
    codes, s, z = co.quantize_rtn(W, bits)
    Y = co.gemm(X, codes, s, z)
    hand = np.zeros((M, N))
    for m in range(M):
        for n in range(N):
            acc = Fraction(0)
            for k in range(128):
                acc += (Fraction(float(X[m, k])) * Fraction(float(s[0, n])) *
                        (int(codes[k, n]) - int(z[0, n])))
            hand[m, n] = float(acc)
    assert np.allclose(Y, hand, rtol=1e-13, atol=1e-15)
    assert np.allclose(Y, X.astype(np.float64) @ rn.dequant(codes, s, z), rtol=1e-13,
                       atol=1e-15)
    cols = np.arange(N)[::-1].copy()
    assert np.array_equal(co.gemm_columns(X, codes, s, z, cols), Y[:, cols])


def test_dropped_zero_point_is_caught_by_one_hot():
    """A planted mistake (w_hat = s * q, z dropped) must disagree with the hand-expanded row."""
    W = inputs.weights(128, 16, seed=21)
    codes, s, z = co.quantize_rtn(W, 3)
    assert np.any(z > 0)
    wrong = s.astype(np.float64) * codes[7].astype(np.float64)
    right = co.dequant(codes, s, z)[7]
    assert not np.array_equal(wrong[0], right)


def test_bad_arguments_are_rejected():
    W = np.zeros((128, 16), np.float16)
    with pytest.raises(ValueError):
        co.quantize_rtn(W, 5)
    with pytest.raises(ValueError):
        co.quantize_rtn(np.zeros((100, 16), np.float16), 3)
    with pytest.raises(ValueError):
        co.pack(np.zeros((128, 10), np.uint8), 3)


@pytest.mark.parametrize("bits", [3, 4])
def test_threaded_gemm_is_the_plain_gemm(bits):
    """The oracle's all-cores GEMM (output columns split over threads, each column its own
    k-ascending sum) equals the single-threaded definition bit for bit, on a ragged N."""
    W = inputs.weights(384, 16 * 37 + 8, seed=bits)
    X = inputs.activations(3, 384, seed=bits)
    codes, s, z = co.quantize_rtn(W, bits)
    assert np.array_equal(co.gemm_threads(X, codes, s, z), co.gemm(X, codes, s, z))


@pytest.mark.parametrize("bits", [3, 4])
def test_threaded_quantizer_is_the_plain_quantizer(bits):
    """The oracle's all-cores quantizer (columns split over threads, each (group, column) by the
    same routine) gives the single-threaded codes, scales and zeros bit for bit, on a ragged N
    with constant and one-signed groups planted."""
    W = inputs.weights(512, 16 * 21 + 8, seed=bits + 10)
    W[:128, 3] = np.float16(0.25)          # a constant group
    W[128:256, 7] = np.abs(W[128:256, 7])  # a one-signed group
    a = co.quantize_rtn(W, bits)
    b = co.quantize_rtn_threads(W, bits)
    for x, y in zip(a, b):
        assert np.array_equal(np.asarray(x).view(np.uint8), np.asarray(y).view(np.uint8))
