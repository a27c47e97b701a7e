"""A lane-level emulation of the planned pass's consumer warps (no GPU).

Where ``test_pass_plan`` walks the plan at the level of records, this walks it lane by lane as
``pass_consumer`` does: each lane (R, c) builds its A fragments from the record's codes and its
B fragments from the staged X (x of batch row R / GPA for the lanes of block record R % GPA,
zeros otherwise), the m16n8k16 MMA is applied as the 16 x 16 by 16 x 8 product its fragments
describe (the public PTX fragment layout), each lane keeps the scale/zero row pairs of the stream
record (packed as the gather kernel packs them) for its two accumulator columns, applies the
block epilogue to its four accumulator values, and at a segment's end the lanes of one output
row add up their batch row's values and write the slot.  The slots are then reduced per local
tile as the kernel does, and Y must match the oracle's fp64 product.
"""
import numpy as np
import pytest

from oracle import c_oracle as co
from paper_2605_08755_gb300 import _lib, inputs
from tests.test_pass_plan import addr, fake_entries, parse, row_offsets


@pytest.fixture(scope="module")
def L():
    from paper_2605_08755_gb300 import build
    build.build()
    return _lib.lib()


def f16_bits(v):
    return int(np.float16(v).view(np.uint16))


def bits_f16(u):
    return float(np.uint16(u).view(np.float16))


def stream_sz(s_col, z_col):
    """The 48-byte scale/zero area of a stream record, as the gather kernel writes it: 32-bit
    word r holds the scales of tile columns r (low half) and r + 8 (high half), 16-bit word r
    the zeros of columns r (low byte) and r + 8 (high byte)."""
    sw = [f16_bits(s_col[r]) | (f16_bits(s_col[r + 8]) << 16) for r in range(8)]
    zw = [int(z_col[r]) | (int(z_col[r + 8]) << 8) for r in range(8)]
    return sw, zw


def a_frags(codes, g, t, cvec):
    """A fragments of every lane for the 8 k16 steps of record (t, g): lane 4R + c holds, for
    step j, a0 = (row R, k = 32c + 4j + e), a1 = (row R + 8, same k), a2 = (row R,
    k = 32c + 4j + 2 + e), a3 = (row R + 8, same k), e = 0, 1, each value c_k + q."""
    q = codes[128 * g:128 * g + 128, 16 * t:16 * t + 16].astype(np.float64)
    val = cvec[:, None] + q                                    # [k, column]
    A = np.zeros((32, 8, 4, 2))
    for lane in range(32):
        R, c = lane >> 2, lane & 3
        for j in range(8):
            for e in range(2):
                k0, k2 = 32 * c + 4 * j + e, 32 * c + 4 * j + 2 + e
                A[lane, j, 0, e] = val[k0, R]
                A[lane, j, 1, e] = val[k0, R + 8]
                A[lane, j, 2, e] = val[k2, R]
                A[lane, j, 3, e] = val[k2, R + 8]
    return A


def mma(D, A, B):
    """D[lane][0..3] += the m16n8k16 product of the warp's fragments.  Matrix A[16][16]: row
    R (a0, a2) and R + 8 (a1, a3), column 2c + e (a0, a1) and 2c + 8 + e (a2, a3); B[16][8]:
    row 2c + e (b0) and 2c + 8 + e (b1), column R; D: rows R (d0, d1) and R + 8 (d2, d3), columns
    2c and 2c + 1."""
    Am = np.zeros((16, 16))
    Bm = np.zeros((16, 8))
    for lane in range(32):
        R, c = lane >> 2, lane & 3
        for e in range(2):
            Am[R, 2 * c + e] = A[lane, 0, e]
            Am[R + 8, 2 * c + e] = A[lane, 1, e]
            Am[R, 2 * c + 8 + e] = A[lane, 2, e]
            Am[R + 8, 2 * c + 8 + e] = A[lane, 3, e]
            Bm[2 * c + e, R] = B[lane, 0, e]
            Bm[2 * c + 8 + e, R] = B[lane, 1, e]
    Dm = Am @ Bm
    for lane in range(32):
        R, c = lane >> 2, lane & 3
        D[lane, 0] += Dm[R, 2 * c]
        D[lane, 1] += Dm[R, 2 * c + 1]
        D[lane, 2] += Dm[R + 8, 2 * c]
        D[lane, 3] += Dm[R + 8, 2 * c + 1]


def emulate_lanes(tb, shapes, bits, data):
    h = tb["h"]
    P, S, M, XR = int(h["sms"]), int(h["nstages"]), int(h["M"]), int(h["xg_row"])
    MP = 1 if M == 1 else 2 if M == 2 else 4
    GPA, LPB = 8 // MP, 4 // MP
    G = [K // 128 for K, _, _ in shapes]
    cvec = row_offsets(bits)
    x_of = {addr(e, "X"): e for e in range(len(shapes))}
    Y = [np.full((M, N), np.nan) for _, N, _ in shapes]
    lanes = np.arange(32)
    Rl, cl = lanes >> 2, lanes & 3
    bl, gil = Rl // GPA, Rl % GPA
    for j in range(P):
        base = int(tb["sm"][j]["rec0"])
        for s in range(S):
            d = tb["stage"][j * S + s]
            n = int(d["n"])
            if n == 0:
                continue
            xs = np.full((M, XR * 128), np.nan)
            for it in tb["x"][int(d["x0"]):int(d["x0"] + d["nx"])]:
                e = x_of[int(it["x"])]
                xs[:, 128 * int(it["xg"]):128 * int(it["xg"]) + int(it["K"])] = data[e][0]
            xg3 = xs.reshape(M, XR, 128)
            sp = np.stack([xg3.sum(2), xg3 @ cvec], 2)
            slots = np.full((int(d["nseg"]), MP, 16), np.nan)
            seg0, wseg = int(d["seg0"]), d["wseg"]
            nr, q_, rem = int(d["nr"]), n // 16, n % 16
            for w in range(16):
                ln = q_ + (1 if w < rem else 0)
                k, k1 = int(wseg[w]), int(wseg[w + 1])
                i = gi = 0
                D = np.zeros((32, 4))
                y = np.zeros((32, 4))
                sw = np.zeros((32, 2), dtype=np.int64)
                zw = np.zeros((32, 2), dtype=np.int64)
                for r in range(nr):
                    if r >= ln:
                        continue
                    sg = tb["seg"][seg0 + k]
                    gr = tb["gather"][base + 16 * r + w]
                    e, rid = int(gr["e"]), int(gr["rid"])
                    t, gg = divmod(rid, G[e])
                    codes, sc, zc = data[e][1], data[e][2], data[e][3]
                    g = int(sg["g0"]) + i
                    A = a_frags(codes, gg, t, cvec)
                    B = np.zeros((32, 8, 2, 2))
                    for lane in range(32):
                        if gil[lane] == gi and bl[lane] < M:
                            xrow = xs[bl[lane], 128 * (int(sg["xg"]) + g):][:128]
                            c = cl[lane]
                            for jj in range(8):
                                B[lane, jj, 0] = xrow[32 * c + 4 * jj:32 * c + 4 * jj + 2]
                                B[lane, jj, 1] = xrow[32 * c + 4 * jj + 2:32 * c + 4 * jj + 4]
                    for jj in range(8):
                        mma(D, A[:, jj], B[:, jj])
                    swr, zwr = stream_sz(sc[gg, 16 * t:16 * t + 16], zc[gg, 16 * t:16 * t + 16])
                    for lane in range(32):
                        c, R = cl[lane], Rl[lane]
                        u0, u1 = (2 * c) % GPA == gi, (2 * c + 1) % GPA == gi
                        if u0 or u1:
                            u = 1 if u1 else 0
                            sw[lane, u], zw[lane, u] = swr[R], zwr[R]
                    i += 1
                    if gi == GPA - 1 or i == int(sg["ng"]):
                        gb = int(sg["xg"]) + int(sg["g0"]) + i - 1 - gi
                        for lane in range(32):
                            c = cl[lane]
                            for v in range(4):
                                col = 2 * c + (v & 1)
                                b, giv = col // GPA, col % GPA
                                if giv <= gi and b < M:
                                    S_, P_ = sp[b, gb + giv]
                                    scv = bits_f16((sw[lane, v & 1] >> (16 * (v >> 1))) & 0xffff)
                                    zcv = float((zw[lane, v & 1] >> (8 * (v >> 1))) & 0xff)
                                    y[lane, v] += scv * (D[lane, v] - P_ - zcv * S_)
                        D[:] = 0
                        gi = 0
                    else:
                        gi += 1
                    if i == int(sg["ng"]):
                        lo = y[:, 0] + y[:, 1]
                        hi = y[:, 2] + y[:, 3]
                        o = 1
                        while o < LPB:  # xor shuffles within the LPB lanes of a batch row
                            lo = lo + lo[lanes ^ o]
                            hi = hi + hi[lanes ^ o]
                            o <<= 1
                        for lane in range(32):
                            c, R = cl[lane], Rl[lane]
                            b = c // LPB
                            if c % LPB == 0 and b < M:
                                slots[k, b, R] = lo[lane]
                                slots[k, b, R + 8] = hi[lane]
                        y[:] = 0
                        k += 1
                        i = 0
                assert k == k1
            for ti in tb["tile"][int(d["tile0"]):int(d["tile0"] + d["nt"])]:
                e = next(e for e in range(len(shapes))
                         if addr(e, "Y") <= int(ti["y"]) < addr(e, "Y") + 2 * shapes[e][1])
                t = (int(ti["y"]) - addr(e, "Y")) // 32
                k0, nk = int(ti["slot0"]), int(ti["nslot"])
                Y[e][:, 16 * t:16 * t + 16] = slots[k0:k0 + nk, :M].sum(0)
            base += n
    return Y


SHAPES = [(256, 32, 0), (1152, 48, 0), (384, 16, 1), (128, 64, 1)]


@pytest.mark.parametrize("bits,M,P", [(3, 1, 2), (4, 1, 3), (3, 2, 2), (4, 3, 2), (3, 4, 1)])
def test_lane_level_consumer_reproduces_the_oracle(L, bits, M, P):
    plan, _ = _lib.pass_plan(fake_entries(SHAPES, bits, M), len(SHAPES), P)
    tb = parse(plan)
    data, refs = [], []
    for e, (K, N, _) in enumerate(SHAPES):
        W = inputs.weights(K, N, seed=800 + e)
        codes, s, z = co.quantize_rtn(W, bits)
        x = inputs.activations(M, K, seed=900 + e)
        # x as the kernel sees it: fp16 values, exactly representable in float64
        data.append((x.astype(np.float64), codes, s.astype(np.float64), z))
        refs.append(co.gemm(x, codes, s, z))
    Y = emulate_lanes(tb, SHAPES, bits, data)
    for e in range(len(SHAPES)):
        assert np.all(np.isfinite(Y[e])), e
        assert np.max(np.abs(Y[e] - refs[e])) <= 1e-9 * (1 + np.max(np.abs(refs[e]))), e
