"""Pins of the pairwise-rotation oracle (oracle/rotation.py) against facts that hold for any
product of Givens rotations: the identity at zero angles, a hand-computed pair, preserved group
norms, the inverse, composition of angles, and the same transform built as an explicit dense
matrix.  CPU only."""
import math

import numpy as np
import pytest

from oracle import rotation as rot
from paper_2605_08755_gb300 import inputs

RNG = np.random.default_rng(77)


def adjacent_pairs(G, R):
    p = np.arange(128, dtype=np.uint8).reshape(64, 2)
    return np.broadcast_to(p, (G, R, 64, 2)).copy()


def test_zero_angles_and_unit_scale_are_the_identity():
    x = RNG.standard_normal((3, 256)).astype(np.float16)
    pairs, _, _ = inputs.rotation(256, 4, seed=1)
    y = rot.pairwise_rotate(x, None, pairs, np.zeros((2, 4, 64), np.float32))
    assert np.array_equal(y, x)


def test_scale_only():
    x = RNG.standard_normal((2, 128)).astype(np.float16)
    a = inputs.rotation(128, 1, seed=2)[2]
    y = rot.pairwise_rotate(x, a, adjacent_pairs(1, 1), np.zeros((1, 1, 64), np.float32))
    assert np.array_equal(y, (x.astype(np.float64) * a.astype(np.float64)).astype(np.float16))


def test_hand_computed_pairs():
    # pair (0, 1) turned by pi/2: (x0, x1) -> (-x1, x0); pair (2, 3) by pi/3; the rest by 0
    x = np.zeros(128)
    x[:4] = [1.0, 2.0, 3.0, 4.0]
    x[4:] = RNG.standard_normal(124)
    th = np.zeros((1, 1, 64))
    th[0, 0, 0] = math.pi / 2
    th[0, 0, 1] = math.pi / 3
    y = rot.pairwise_rotate64(x, None, adjacent_pairs(1, 1), th)[0]
    c, s = 0.5, math.sqrt(3) / 2
    assert np.allclose(y[:4], [-2.0, 1.0, 3 * c - 4 * s, 3 * s + 4 * c], rtol=0, atol=1e-15)
    assert np.array_equal(y[4:], x[4:])


def test_group_norms_are_preserved_and_groups_do_not_mix():
    x = RNG.standard_normal((4, 384))
    pairs, theta, _ = inputs.rotation(384, 8, seed=3)
    y = rot.pairwise_rotate64(x, None, pairs, theta)
    for g in range(3):
        sl = slice(128 * g, 128 * (g + 1))
        assert np.allclose(np.linalg.norm(y[:, sl], axis=1), np.linalg.norm(x[:, sl], axis=1),
                           rtol=1e-13)
    # a change in group 0 leaves groups 1 and 2 alone
    x2 = x.copy()
    x2[:, 5] += 1.0
    y2 = rot.pairwise_rotate64(x2, None, pairs, theta)
    assert np.array_equal(y2[:, 128:], y[:, 128:])
    assert not np.array_equal(y2[:, :128], y[:, :128])


def test_the_inverse_undoes_it():
    x = RNG.standard_normal((2, 256))
    pairs, theta, _ = inputs.rotation(256, 6, seed=4)
    y = rot.pairwise_rotate64(x, None, pairs, theta)
    back = rot.pairwise_rotate64(y, None, pairs[:, ::-1], -theta[:, ::-1])
    assert np.allclose(back, x, rtol=0, atol=1e-13)


def test_angles_on_the_same_pairs_add():
    x = RNG.standard_normal((2, 128))
    pairs = np.repeat(inputs.rotation(128, 1, seed=5)[0], 2, axis=1)  # one matching, twice
    t = RNG.uniform(-3, 3, (1, 2, 64))
    two = rot.pairwise_rotate64(x, None, pairs, t)
    one = rot.pairwise_rotate64(x, None, pairs[:, :1], t.sum(axis=1, keepdims=True))
    assert np.allclose(two, one, rtol=0, atol=1e-13)


def test_equals_the_dense_product_of_givens_matrices():
    # v' = v @ Q with Q = diag(alpha) @ G_0 @ G_1 @ ... (rounds applied in order); each G_r is
    # built entry by entry from its pairs
    K, R = 256, 3
    pairs, theta, alpha = inputs.rotation(K, R, seed=6)
    Q = np.diag(alpha.astype(np.float64))
    for r in range(R):
        Gr = np.eye(K)
        for g in range(K // 128):
            for p in range(64):
                i, j = 128 * g + int(pairs[g, r, p, 0]), 128 * g + int(pairs[g, r, p, 1])
                c, s = math.cos(theta[g, r, p]), math.sin(theta[g, r, p])
                Gr[i, i], Gr[j, i], Gr[i, j], Gr[j, j] = c, -s, s, c
        Q = Q @ Gr
    x = RNG.standard_normal((3, K)).astype(np.float16)
    ref = x.astype(np.float64) @ Q
    assert np.allclose(rot.pairwise_rotate64(x, alpha, pairs, theta), ref, rtol=0, atol=1e-12)


def test_rejects_a_round_that_is_not_a_matching():
    pairs = adjacent_pairs(1, 1)
    pairs[0, 0, 1, 0] = 0  # channel 0 twice, channel 2 never
    with pytest.raises(ValueError):
        rot.pairwise_rotate(np.zeros((1, 128)), None, pairs, np.zeros((1, 1, 64)))
