"""CPU oracle for an online pairwise rotation of a projection's input (numpy, float64).

TEST INFRASTRUCTURE ONLY (like the rest of ``oracle``): the tests, ``smoke()`` and the
benchmark's CPU leg may use it; the product path never does.  It shares no code with the CUDA
library.

The paper sets LAQuant against rotation-based methods whose transform of the activations cannot
be folded into the weights and so runs at every forward pass (Sec. 1 and Sec. 2; ParoQuant:
pairwise rotations with channel scaling), and Sec. 5.2 measures the decode speed gained by not
running it.  The paper does not define the transform.  The reading restated here:

* the K input channels of a projection fall into groups of 128 (the quantization groups);
* the row vector x is first scaled per channel, v = x * alpha;
* then ``rounds`` rounds of Givens rotations run in order; round r of group g holds 64 pairs
  (i, j) of the group's channels that partition it, each with an angle t, and maps
  (v_i, v_j) -> (v_i cos t - v_j sin t, v_i sin t + v_j cos t);
* the result is rounded to fp16 once.
"""
import numpy as np


def _check_matching(pairs):
    """Every round of every group must pair up the group's 128 channels exactly once."""
    G, R = pairs.shape[:2]
    for g in range(G):
        for r in range(R):
            if sorted(int(c) for c in pairs[g, r].reshape(-1)) != list(range(128)):
                raise ValueError(f"round {r} of group {g} is not a perfect matching of 0..127")


def pairwise_rotate64(x, alpha, pairs, theta):
    """x [M, K] (any float type), alpha [K] or None, pairs uint8 [K/128, R, 64, 2], theta
    [K/128, R, 64] -> float64 [M, K]: the transform above without the final rounding."""
    v = np.array(np.asarray(x), dtype=np.float64, copy=True)
    if v.ndim == 1:
        v = v[None, :]
    M, K = v.shape
    pairs = np.asarray(pairs)
    theta = np.asarray(theta, dtype=np.float64)
    G, R = pairs.shape[:2]
    if K != 128 * G or theta.shape != (G, R, 64):
        raise ValueError("table shapes do not match K")
    _check_matching(pairs)
    if alpha is not None:
        v *= np.asarray(alpha, dtype=np.float64)[None, :]
    for g in range(G):
        base = 128 * g
        for r in range(R):
            for p in range(64):
                i = base + int(pairs[g, r, p, 0])
                j = base + int(pairs[g, r, p, 1])
                c, s = np.cos(theta[g, r, p]), np.sin(theta[g, r, p])
                vi, vj = v[:, i].copy(), v[:, j].copy()
                v[:, i] = vi * c - vj * s
                v[:, j] = vi * s + vj * c
    return v


def pairwise_rotate(x, alpha, pairs, theta):
    """The transform rounded to fp16 once: fp16 [M, K]."""
    return pairwise_rotate64(x, alpha, pairs, theta).astype(np.float16)
