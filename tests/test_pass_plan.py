"""Host-side checks of the planned pass (laq_pass_*; no GPU): the plan's tables parsed with numpy
and checked against what the planner promises, and an emulation that walks the tables exactly as
the kernel does (rounds, warp positions, segments, blocks of eight groups, slots, local tiles),
taking every record's codes from the stream the gather table describes, and reproduces the
oracle's Y.  The kernel itself runs only on a GPU."""
import ctypes

import numpy as np
import pytest

from oracle import c_oracle as co
from paper_2605_08755_gb300 import _lib, inputs

HDR = np.dtype([("magic", "<u4"), ("version", "<i4"), ("count", "<i4"), ("nstages", "<i4"),
                ("sms", "<i4"), ("bits", "<i4"), ("rb", "<i4"), ("M", "<i4"),
                ("xg_row", "<i4"), ("xs_bytes", "<i4"),
                ("max_segs", "<i4"), ("max_nx", "<i4"), ("records", "<i8"), ("rounds", "<i8"),
                ("segs", "<i8"), ("ltiles", "<i8"), ("xitems", "<i8"), ("tables_h", "<i8"),
                ("tables_bytes", "<i8"), ("stream_bytes", "<i8"), ("o_sm", "<i8"),
                ("o_rounds", "<i8"), ("o_stage", "<i8"), ("o_seg", "<i8"), ("o_tile", "<i8"),
                ("o_x", "<i8"), ("o_prep", "<i8"), ("o_gather", "<i8"), ("plan_bytes", "<i8"),
                ("device_bytes", "<i8")])
SM = np.dtype([("rec0", "<i8"), ("round0", "<i4"), ("nrounds", "<i4")])
STAGE = np.dtype([("n", "<i4"), ("nr", "<i4"), ("seg0", "<i4"), ("tile0", "<i4"), ("x0", "<i4"),
                  ("nseg", "<i2"), ("nt", "<i2"), ("nx", "<i2"), ("pad", "<i2"),
                  ("wseg", "u1", (17,)), ("pad2", "u1", (3,))])
SEG = np.dtype([("e", "<i4"), ("t", "<i4"), ("g0", "<i2"), ("ng", "<i2"), ("xg", "<i2"),
                ("lt", "<i2")])
TILE = np.dtype([("y", "<u8"), ("slot0", "<i4"), ("nslot", "<i4"), ("ldy", "<i4"),
                 ("pad", "<i4")])
XIT = np.dtype([("x", "<u8"), ("K", "<i4"), ("xg", "<i4")])
PREP = np.dtype([("packed", "<u8"), ("s", "<u8"), ("z", "<u8"), ("N", "<i4"), ("G", "<i4")])
GATHER = np.dtype([("e", "<i4"), ("rid", "<i4")])

MiB = 1 << 20


@pytest.fixture(scope="module")
def L():
    from paper_2605_08755_gb300 import build
    build.build()
    return _lib.lib()


def fake_entries(shapes, bits=3, M=1):
    """laq_gemv entries with distinct, 16-byte aligned fake device addresses (never touched by
    the host-only planner).  ``shapes``: (K, N, wait_prev) per entry."""
    arr = (_lib.Gemv * max(1, len(shapes)))()
    for i, (K, N, wait) in enumerate(shapes):
        base = (i + 1) * 64 * MiB
        arr[i] = _lib.Gemv(base, base + 8 * MiB, base + 16 * MiB, base + 24 * MiB,
                           base + 32 * MiB, M, K, N, bits, wait)
    return arr


def addr(i, what):
    return (i + 1) * 64 * MiB + {"X": 0, "packed": 8, "s": 16, "z": 24, "Y": 32}[what] * MiB


def parse(plan):
    buf = np.frombuffer(plan, dtype=np.uint8)
    h = buf[:HDR.itemsize].view(HDR)[0]
    t = buf[int(h["tables_h"]):int(h["tables_h"] + h["tables_bytes"])]

    def tab(off, dt, n):
        return t[int(off):int(off) + int(n) * dt.itemsize].view(dt)
    return {
        "h": h,
        "sm": tab(h["o_sm"], SM, h["sms"]),
        "rounds": t[int(h["o_rounds"]):int(h["o_rounds"] + h["rounds"])],
        "stage": tab(h["o_stage"], STAGE, int(h["sms"]) * int(h["nstages"])),
        "seg": tab(h["o_seg"], SEG, h["segs"]),
        "tile": tab(h["o_tile"], TILE, h["ltiles"]),
        "x": tab(h["o_x"], XIT, h["xitems"]),
        "prep": tab(h["o_prep"], PREP, h["count"]),
        "gather": tab(h["o_gather"], GATHER, h["records"]),
    }


def stage_starts(shapes):
    return [i for i, (_, _, w) in enumerate(shapes) if i == 0 or w]


def warp_records(tb, seg0, wseg, w):
    """Warp w's records of an (SM, stage) in order: (e, t, g, segment index, xg)."""
    out = []
    for k in range(int(wseg[w]), int(wseg[w + 1])):
        s = tb["seg"][seg0 + k]
        for i in range(int(s["ng"])):
            out.append((int(s["e"]), int(s["t"]), int(s["g0"]) + i, k, int(s["xg"])))
    return out


def check_plan(shapes, P, bits, plan, dev_bytes, M=1):
    """Every promise of the plan, checked from its tables."""
    tb = parse(plan)
    h = tb["h"]
    assert h["M"] == M
    S = len(stage_starts(shapes))
    starts = stage_starts(shapes) + [len(shapes)]
    rb = (1024 if bits == 4 else 768) + 48
    assert h["magic"] == 0x5051414C and h["count"] == len(shapes) and h["nstages"] == S
    assert h["sms"] == P and h["bits"] == bits and h["rb"] == rb
    assert h["device_bytes"] == dev_bytes == h["stream_bytes"] + h["tables_bytes"]
    assert h["stream_bytes"] == -(-int(h["records"]) * rb // 256) * 256
    # the gather table is a permutation of every entry's records
    G = [K // 128 for K, _, _ in shapes]
    T = [N // 16 for _, N, _ in shapes]
    gat = tb["gather"]
    assert len(gat) == sum(g * t for g, t in zip(G, T))
    key = gat["e"].astype(np.int64) * (1 << 32) + gat["rid"]
    want = np.concatenate([e * (1 << 32) + np.arange(G[e] * T[e], dtype=np.int64)
                           for e in range(len(shapes))]) if shapes else np.zeros(0, np.int64)
    assert np.array_equal(np.sort(key), np.sort(want))
    for e, pe in enumerate(tb["prep"]):
        assert (pe["packed"], pe["s"], pe["z"], pe["N"], pe["G"]) == (
            addr(e, "packed"), addr(e, "s"), addr(e, "z"), shapes[e][1], G[e])
    owner = {}  # (e, t) -> SM
    xs_max = segs_max = nx_max = 0
    rec = 0
    for j in range(P):
        sm = tb["sm"][j]
        assert sm["rec0"] == rec
        rnds = tb["rounds"][int(sm["round0"]):int(sm["round0"] + sm["nrounds"])]
        r_at = 0
        for s in range(S):
            d = tb["stage"][j * S + s]
            n, nr = int(d["n"]), int(d["nr"])
            assert nr == -(-n // 16)
            q, rem = divmod(n, 16)
            assert list(rnds[r_at:r_at + nr]) == [16] * q + ([rem] if rem else [])
            r_at += nr
            if n == 0:
                continue
            seg0, nseg, wseg = int(d["seg0"]), int(d["nseg"]), d["wseg"]
            assert wseg[0] == 0 and wseg[16] == nseg and np.all(np.diff(wseg.astype(int)) >= 0)
            segs_max = max(segs_max, nseg)
            lists = [warp_records(tb, seg0, wseg, w) for w in range(16)]
            assert [len(x) for x in lists] == [q + (w < rem) for w in range(16)]
            recs = [r for x in lists for r in x]
            # whole tiles of this stage, every group once, in order
            tiles = []
            for (e, t, g, k, xg) in recs:
                assert starts[s] <= e < starts[s + 1]
                if not tiles or tiles[-1] != (e, t):
                    tiles.append((e, t))
                    assert g == 0
            for (e, t) in tiles:
                assert (e, t) not in owner
                owner[(e, t)] = j
                assert sum(1 for r in recs if r[:2] == (e, t)) == G[e]
            # local tiles: Y address and the contiguous segments covering each
            assert int(d["nt"]) == len(tiles)
            for lt, (e, t) in enumerate(tiles):
                ti = tb["tile"][int(d["tile0"]) + lt]
                assert ti["y"] == addr(e, "Y") + 32 * t and ti["ldy"] == shapes[e][1]
                ks = sorted({r[3] for r in recs if r[:2] == (e, t)})
                assert ks == list(range(int(ti["slot0"]), int(ti["slot0"] + ti["nslot"])))
                assert all(int(tb["seg"][seg0 + k]["lt"]) == lt for k in ks)
            # staged X: each touched entry once, whole groups one after another
            xi = tb["x"][int(d["x0"]):int(d["x0"] + d["nx"])]
            ents = sorted({e for e, _ in tiles})
            assert [addr(e, "X") for e in ents] == [int(v) for v in xi["x"]]
            assert list(xi["K"]) == [shapes[e][0] for e in ents]
            assert list(xi["xg"]) == list(np.cumsum([0] + [G[e] for e in ents])[:-1])
            for (e, t, g, k, xg) in recs:
                assert xg == int(xi["xg"][ents.index(e)])
            xs_max = max(xs_max, sum(G[e] for e in ents))
            nx_max = max(nx_max, len(ents))
            # the stream: round r, position w holds warp w's r-th record
            for r in range(nr):
                for w in range(16 if r < q else rem):
                    e, t, g, _, _ = lists[w][r]
                    gr = gat[rec]
                    assert (int(gr["e"]), int(gr["rid"])) == (e, t * G[e] + g)
                    rec += 1
        assert r_at == len(rnds)
    assert rec == len(gat)
    assert len(owner) == sum(T)
    assert (h["xg_row"], h["max_segs"], h["max_nx"]) == (xs_max, segs_max, nx_max)
    assert h["xs_bytes"] == 256 * M * xs_max
    # balance: an SM's share of a stage exceeds the even share by less than one tile
    for s in range(S):
        n = [int(tb["stage"][j * S + s]["n"]) for j in range(P)]
        W = sum(G[e] * T[e] for e in range(starts[s], starts[s + 1]))
        gmax = max(G[e] for e in range(starts[s], starts[s + 1]))
        assert max(n) <= -(-W // P) + gmax
    return tb


def row_offsets(bits):
    """c_k = 2^(10 - p) of the record layout for the 128 rows of a group: row k is pair
    (k % 32) // 2, whose codes sit at mantissa bit p (b = 4: p = 0, 4 alternating; b = 3:
    p = 1 for pairs 0-5, 4 for 6-11, 7 for 12-14, 4 for pair 15)."""
    pair = (np.arange(128) % 32) // 2
    if bits == 4:
        return np.where(pair % 2 == 1, 64.0, 1024.0)
    return np.select([pair < 6, pair < 12, pair < 15], [512.0, 64.0, 8.0], 64.0)


def emulate(tb, shapes, bits, data):
    """Y of every entry, computed by walking the plan as the kernel does, in float64.
    ``data[e]`` = (x [M, K] float64, codes [K, N], s [G, N] float64, z [G, N]).  Each record's
    codes, scales and zeros come from the stream record the gather table puts at the warp's
    position of its round; its x from the warp's own segment, in the X area whose rows are
    xg_row groups apart; blocks hold 8 / MP records (MP = M rounded up to 1, 2, 4) and the block
    epilogue uses the kernel's indices (the block's first group gb, MMA column = batch row b and
    block record giv) and Eq. (1) in the kernel's form y += s (D - P - z S) with
    D = sum_k (c_k + q_k) x_k; slots hold one row of 16 outputs per (segment, batch row)."""
    h = tb["h"]
    P, S, M, XR = int(h["sms"]), int(h["nstages"]), int(h["M"]), int(h["xg_row"])
    MP = 1 if M == 1 else 2 if M == 2 else 4
    GPA = 8 // MP
    G = [K // 128 for K, _, _ in shapes]
    c = row_offsets(bits)
    x_of = {addr(e, "X"): e for e in range(len(shapes))}
    Y = [np.full((M, N), np.nan) for _, N, _ in shapes]
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
            sp = np.stack([xg3.sum(2), xg3 @ c], 2)  # (S, P) per (row, staged group)
            slots = np.full((int(d["nseg"]), MP, 16), np.nan)
            seg0, wseg = int(d["seg0"]), d["wseg"]
            for w in range(16):
                r = 0
                for k in range(int(wseg[w]), int(wseg[w + 1])):
                    sg = tb["seg"][seg0 + k]
                    ng, g0, xg = int(sg["ng"]), int(sg["g0"]), int(sg["xg"])
                    y = np.zeros((M, 16))
                    i = gi = 0
                    Dcol, scol, zcol = {}, {}, {}
                    while i < ng:
                        gr = tb["gather"][base + 16 * r + w]  # round r, position w
                        e, rid = int(gr["e"]), int(gr["rid"])
                        t, g = divmod(rid, G[e])
                        codes, sc, zc = data[e][1], data[e][2], data[e][3]
                        q = codes[128 * g:128 * g + 128, 16 * t:16 * t + 16].astype(np.float64)
                        for b in range(M):  # MMA column b * GPA + gi
                            x = xs[b, 128 * (xg + g0 + i):128 * (xg + g0 + i) + 128]
                            Dcol[b, gi] = (c[:, None] + q).T @ x
                        scol[gi] = sc[g, 16 * t:16 * t + 16]
                        zcol[gi] = zc[g, 16 * t:16 * t + 16].astype(np.float64)
                        i += 1
                        r += 1
                        if gi == GPA - 1 or i == ng:
                            gb = xg + g0 + i - 1 - gi
                            for b in range(M):
                                for giv in range(gi + 1):
                                    S_, P_ = sp[b, gb + giv]
                                    y[b] += scol[giv] * (Dcol[b, giv] - P_ - zcol[giv] * S_)
                            gi = 0
                        else:
                            gi += 1
                    slots[k, :M] = y
            for ti in tb["tile"][int(d["tile0"]):int(d["tile0"] + d["nt"])]:
                e = next(e for e in range(len(shapes))
                         if addr(e, "Y") <= int(ti["y"]) < addr(e, "Y") + 2 * shapes[e][1])
                assert int(ti["ldy"]) == shapes[e][1]
                t = (int(ti["y"]) - addr(e, "Y")) // 32
                k0, nk = int(ti["slot0"]), int(ti["nslot"])
                Y[e][:, 16 * t:16 * t + 16] = slots[k0:k0 + nk, :M].sum(0)
            base += n
    return Y


SMALL = [(256, 48, 0), (384, 32, 0), (128, 16, 1), (1024, 160, 1), (256, 64, 0), (640, 16, 1),
         (128, 512, 1), (1024, 32, 1), (2048, 16, 0)]


@pytest.mark.parametrize("bits,P,M", [(3, 5, 1), (4, 7, 1), (3, 1, 1), (4, 3, 1), (3, 5, 2),
                                      (4, 3, 3), (3, 7, 4)])
def test_plan_emulation_reproduces_the_oracle(L, bits, P, M):
    arr = fake_entries(SMALL, bits, M)
    plan, dev = _lib.pass_plan(arr, len(SMALL), P)
    tb = check_plan(SMALL, P, bits, plan, dev, M)
    data, refs = [], []
    for e, (K, N, _) in enumerate(SMALL):
        W = inputs.weights(K, N, seed=300 + e)
        codes, s, z = co.quantize_rtn(W, bits)
        x = inputs.activations(M, K, seed=400 + e)
        data.append((x.astype(np.float64), codes, s.astype(np.float64), z))
        refs.append(co.gemm(x, codes, s, z))
    Y = emulate(tb, SMALL, bits, data)
    for e in range(len(SMALL)):
        assert np.all(np.isfinite(Y[e])), e
        assert np.max(np.abs(Y[e] - refs[e])) <= 1e-9 * (1 + np.max(np.abs(refs[e]))), e


def test_plan_of_the_qwen3_4b_fused_pass(L):
    """Four layers of the fused Qwen3-4B-shaped pass (q|k|v, o, gate|up, down) on 152 SMs,
    W3: every table invariant, and whole tiles (no output tile split between SMs)."""
    shapes = []
    for layer in range(4):
        shapes += [(2560, 6144, 1), (4096, 2560, 1), (2560, 19456, 1), (9728, 2560, 1)]
    arr = fake_entries(shapes, 3)
    plan, dev = _lib.pass_plan(arr, len(shapes), 152)
    tb = check_plan(shapes, 152, 3, plan, dev)
    h = tb["h"]
    assert h["nstages"] == 16 and h["xs_bytes"] == 2 * 9728
    # gate|up: 1216 tiles of 20 records, 8 per SM exactly; down: 160 tiles on 152 SMs
    n_gu = [int(tb["stage"][j * 16 + 2]["n"]) for j in range(152)]
    assert set(n_gu) == {160}
    n_down = sorted(int(tb["stage"][j * 16 + 3]["n"]) for j in range(152))
    assert n_down.count(152) == 8 and n_down.count(76) == 144


def test_plan_of_the_full_qwen3_4b_unfused_pass(L):
    """The 252-entry pass (k, v after q and up after gate share their stage): sizes and the
    gather permutation at full size (36 layers)."""
    shapes = []
    for layer in range(36):
        for name, K, N in inputs.QWEN3_4B:
            shapes.append((K, N, 0 if name in ("k", "v", "up") else 1))
    arr = fake_entries(shapes, 3)
    plan, dev = _lib.pass_plan(arr, len(shapes), 152)
    tb = parse(plan)
    h = tb["h"]
    assert h["count"] == 252 and h["nstages"] == 144
    records = sum((K // 128) * (N // 16) for K, N, _ in shapes)
    assert h["records"] == records and h["stream_bytes"] == -(-records * 816 // 256) * 256
    gat = tb["gather"]
    key = np.sort(gat["e"].astype(np.int64) * (1 << 32) + gat["rid"])
    assert np.all(np.diff(key) > 0)
    counts = np.bincount(gat["e"], minlength=252)
    assert list(counts) == [(K // 128) * (N // 16) for K, N, _ in shapes]
    assert int(tb["sm"]["nrounds"].sum()) == h["rounds"] == int(tb["stage"]["nr"].sum())


def status(f, *a):
    return int(f(*a))


def sizes(L, arr, count, P):
    pb, db = ctypes.c_size_t(0), ctypes.c_size_t(0)
    return int(L.laq_pass_plan_sizes(arr, count, P, ctypes.byref(pb), ctypes.byref(db)))


def test_plan_rejects_invalid_entries(L):
    ok = [(256, 32, 0), (256, 16, 1)]
    assert sizes(L, fake_entries(ok), 2, 4) == 0
    arr = fake_entries(ok)
    arr[1].bits = 4
    assert sizes(L, arr, 2, 4) == 2                              # mixed bits
    arr = fake_entries(ok)
    arr[0].bits = 5
    assert sizes(L, arr, 2, 4) == 2
    assert sizes(L, fake_entries(ok, M=4), 2, 4) == 0
    assert sizes(L, fake_entries(ok, M=5), 2, 4) == 6            # M outside 1..4
    assert sizes(L, fake_entries(ok, M=0), 2, 4) == 6
    arr = fake_entries(ok)
    arr[1].M = 2
    assert sizes(L, arr, 2, 4) == 6                              # mixed M
    assert sizes(L, fake_entries([(13312, 16, 0)], M=4), 1, 4) == 0   # 4 x 13312 x 2 = 104 KB
    assert sizes(L, fake_entries([(13440, 16, 0)], M=4), 1, 4) == 4
    assert sizes(L, fake_entries([(100, 16, 0)]), 1, 4) == 4     # K % 128
    assert sizes(L, fake_entries([(128, 24, 0)]), 1, 4) == 4     # N % 16
    assert sizes(L, fake_entries([(0, 16, 0)]), 1, 4) == 4
    assert sizes(L, fake_entries([(53248, 16, 0)]), 1, 4) == 0   # largest K at M = 1
    assert sizes(L, fake_entries([(53248 + 128, 16, 0)]), 1, 4) == 4
    # 2^23 tiles of 416 groups: record ids t * G + g would pass 2^31
    assert sizes(L, fake_entries([(53248, 16 << 23, 0)]), 1, 4) == 4
    assert sizes(L, fake_entries(ok), 2, 0) == 4                 # no SMs
    assert sizes(L, fake_entries(ok), 2, 1025) == 4
    assert sizes(L, fake_entries([(128, 16, 0)] * 385), 385, 4) == 4
    assert sizes(L, fake_entries([(128, 16, 0)] * 384), 384, 4) == 0
    arr = fake_entries(ok)
    arr[1].Y = None
    assert sizes(L, arr, 2, 4) == 1                              # NULL
    arr = fake_entries(ok)
    arr[0].s = arr[0].s + 2
    assert sizes(L, arr, 2, 4) == 5                              # misaligned
    # two entries of one stage whose X together exceed the staging area on one SM
    assert sizes(L, fake_entries([(32768, 16, 0), (32768, 16, 0)]), 2, 1) == 4
    pb = ctypes.c_size_t(0)
    assert int(L.laq_pass_plan_sizes(fake_entries(ok), 2, 4, None, ctypes.byref(pb))) == 1


def test_plan_buffer_and_run_arguments(L):
    arr = fake_entries([(256, 32, 0), (512, 48, 1)])
    pb, db = ctypes.c_size_t(0), ctypes.c_size_t(0)
    assert L.laq_pass_plan_sizes(arr, 2, 8, ctypes.byref(pb), ctypes.byref(db)) == 0
    small = (ctypes.c_uint8 * (pb.value - 1))()
    assert L.laq_pass_plan_build(arr, 2, 8, small, pb.value - 1) == 10   # LAQ_ERR_WORKSPACE
    assert L.laq_pass_plan_build(arr, 2, 8, None, pb.value) == 1
    plan, dev = _lib.pass_plan(arr, 2, 8)
    assert dev == db.value
    ws = int(L.laq_pass_workspace_bytes(plan))
    assert ws == 1280                      # status and finished count, 8 stage counters (lines)
    junk = (ctypes.c_uint8 * 512)()
    assert L.laq_pass_workspace_bytes(junk) == 0
    assert L.laq_pass_workspace_bytes(None) == 0
    D, WS = ctypes.c_void_p(0x100000), ctypes.c_void_p(0x200000)
    # rejected on the host, before any CUDA call
    assert L.laq_pass_prepare(junk, D, dev, None) == 9                  # not a plan
    assert L.laq_pass_prepare(plan, None, dev, None) == 1
    assert L.laq_pass_prepare(plan, ctypes.c_void_p(0x100010), dev, None) == 5
    assert L.laq_pass_prepare(plan, D, dev - 1, None) == 10
    assert L.laq_pass_run(junk, D, WS, ws, None) == 9
    assert L.laq_pass_run(plan, None, WS, ws, None) == 1
    assert L.laq_pass_run(plan, D, None, ws, None) == 1
    assert L.laq_pass_run(plan, ctypes.c_void_p(0x100080), WS, ws, None) == 5
    assert L.laq_pass_run(plan, D, WS, ws - 248, None) == 10
    assert L.laq_pass_run(plan, D, ctypes.c_void_p(0x200004), ws, None) == 10
    # an empty chain plans to nothing and runs as a no-op
    empty, dev0 = _lib.pass_plan(fake_entries([]), 0, 8)
    assert parse(empty)["h"]["nstages"] == 0 and parse(empty)["h"]["records"] == 0
    assert L.laq_pass_run(empty, D, WS, L.laq_pass_workspace_bytes(empty), None) == 0


def test_segment_limit_per_sm_stage(L):
    """An SM's share of a stage holds at most 255 warp segments (one-group tiles here: a segment
    per tile); one more is rejected with LAQ_ERR_SHAPE."""
    assert sizes(L, fake_entries([(128, 16 * 255, 0)]), 1, 1) == 0
    assert sizes(L, fake_entries([(128, 16 * 256, 0)]), 1, 1) == 4
    plan, dev = _lib.pass_plan(fake_entries([(128, 16 * 255, 0)]), 1, 1)
    tb = check_plan([(128, 16 * 255, 0)], 1, 3, plan, dev)
    assert tb["h"]["max_segs"] == 255
