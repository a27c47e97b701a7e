"""GPU parity of the online pairwise rotation (laq_rotation_tables, laq_pairwise_rotate) against
oracle/rotation.py.

Tolerance per element, from the arithmetic: the kernel scales and rotates in fp32, each Givens
update adding at most about 2 * 2^-24 of its pair's norm and each table entry (sincosf) about
2^-23, so after R rounds the fp32 result is within (4R + 2) * 2^-24 * ||v_g|| of the exact one
(v_g: the scaled group); both sides then round to fp16 once (half an ulp each, 2^-11 relative,
or 2^-25 absolute below fp16's normal range).  So |gpu - ref| <= 2^-10 |ref| +
(4R + 2) 2^-24 ||v_g|| + 2^-24."""
import numpy as np
import pytest

torch = pytest.importorskip("torch")

import paper_2605_08755_gb300 as laq  # noqa: E402
from paper_2605_08755_gb300 import _lib, inputs  # noqa: E402
from oracle import rotation as rot  # noqa: E402

pytestmark = pytest.mark.gpu
DEV = "cuda"
RNG = np.random.default_rng(99)


def dev(a):
    return torch.from_numpy(np.ascontiguousarray(a)).to(DEV)


def host(t):
    torch.cuda.synchronize()
    return t.cpu().numpy()


def check(gpu, x, alpha, pairs, theta):
    ref64 = rot.pairwise_rotate64(x, alpha, pairs, theta)
    ref = ref64.astype(np.float16).astype(np.float64)
    M, K = ref64.shape
    R = pairs.shape[1]
    v = x.astype(np.float64) * (1.0 if alpha is None else alpha.astype(np.float64))
    gnorm = np.linalg.norm(v.reshape(M, K // 128, 128), axis=2)           # [M, G]
    tol = (2.0 ** -10 * np.abs(ref64) + (4 * R + 2) * 2.0 ** -24
           * np.repeat(gnorm, 128, axis=1) + 2.0 ** -24)
    err = np.abs(np.asarray(gpu, np.float64) - ref)
    assert np.all(err <= tol), f"max err {err.max()}, worst ratio {(err / tol).max()}"


def test_rotation_tables_are_cos_and_sin():
    theta = inputs.rotation(2560, 8, seed=1)[1]
    cs = host(_lib.laq_rotation_tables(dev(theta)))
    t = theta.astype(np.float64)
    assert np.abs(cs[..., 0] - np.cos(t)).max() <= 2.0 ** -22
    assert np.abs(cs[..., 1] - np.sin(t)).max() <= 2.0 ** -22


@pytest.mark.parametrize("M", [1, 3, 16])
@pytest.mark.parametrize("K,R", [(128, 1), (2560, 8), (9728, 8), (384, 16), (4096, 4)])
@pytest.mark.parametrize("scaled", [False, True])
def test_rotate_matches_the_oracle(M, K, R, scaled):
    pairs, theta, alpha = inputs.rotation(K, R, seed=K + R)
    x = (RNG.standard_normal((M, K)) * 2).astype(np.float16)
    a = alpha if scaled else None
    Y = _lib.laq_pairwise_rotate(dev(x), dev(pairs), _lib.laq_rotation_tables(dev(theta)),
                                 alpha=dev(a) if scaled else None)
    check(host(Y), x, a, pairs, theta)


def test_in_place_and_ragged_group_count():
    # K / 128 = 7 groups: the last CTA has 3 of its 4 warps busy
    M, K, R = 5, 896, 6
    pairs, theta, alpha = inputs.rotation(K, R, seed=3)
    x = RNG.standard_normal((M, K)).astype(np.float16)
    X = dev(x)
    _lib.laq_pairwise_rotate(X, dev(pairs), _lib.laq_rotation_tables(dev(theta)),
                             alpha=dev(alpha), Y=X)
    check(host(X), x, alpha, pairs, theta)


def test_zero_angles_are_exact():
    # cos 0 = 1, sin 0 = 0 and an fp16 x fp16 product is exact in fp32: bit for bit
    M, K, R = 2, 2560, 8
    pairs, _, alpha = inputs.rotation(K, R, seed=4)
    zero = np.zeros((K // 128, R, 64), np.float32)
    x = RNG.standard_normal((M, K)).astype(np.float16)
    Y = _lib.laq_pairwise_rotate(dev(x), dev(pairs), _lib.laq_rotation_tables(dev(zero)),
                                 alpha=dev(alpha))
    assert np.array_equal(host(Y), rot.pairwise_rotate(x, alpha, pairs, zero))
    Y0 = _lib.laq_pairwise_rotate(dev(x), dev(pairs[:, :0]), dev(np.zeros((K // 128, 0, 64, 2),
                                                                          np.float32)))
    assert np.array_equal(host(Y0), x)  # no rounds, no scales: a copy


def test_empty_and_rejected_arguments():
    K, R = 256, 2
    pairs, theta, _ = inputs.rotation(K, R, seed=5)
    P, CS = dev(pairs), _lib.laq_rotation_tables(dev(theta))
    empty = torch.empty((0, K), dtype=torch.float16, device=DEV)
    assert _lib.laq_pairwise_rotate(empty, P, CS).shape == (0, K)
    x = torch.zeros((1, K), dtype=torch.float16, device=DEV)
    L = _lib.lib()
    st = L.laq_pairwise_rotate(_lib._ptr(x), 1, 200, None, _lib._ptr(P), _lib._ptr(CS), R,
                               _lib._ptr(x), _lib._stream(None))
    assert st == 4  # LAQ_ERR_SHAPE: K not a multiple of 128
    st = L.laq_pairwise_rotate(_lib._ptr(x), 1, K, None, _lib._ptr(P), _lib._ptr(CS), 17,
                               _lib._ptr(x), _lib._stream(None))
    assert st == 4  # more than 16 rounds
    flat = torch.zeros(K + 8, dtype=torch.float16, device=DEV)
    st = L.laq_pairwise_rotate(_lib._ptr(flat[4:]), 1, K, None, _lib._ptr(P), _lib._ptr(CS), R,
                               _lib._ptr(flat[4:]), _lib._stream(None))
    assert st == 5  # LAQ_ERR_ALIGN: X 8 bytes off a 16-byte boundary
    with pytest.raises(laq.LaqError):
        _lib.laq_pairwise_rotate(x, P, CS, alpha=flat[4:4 + K])
