"""Independent numpy (float64) restatement of the oracle, for cross-checking the C oracle.

TEST INFRASTRUCTURE ONLY.  Written separately from ``laq_oracle.c`` (vectorised library calls
instead of loops) so that a slip in one shows up as a mismatch against the other.

* ``quantize_rtn`` -- Eq. (1) of LAQuant with min-max RTN initialisation: zero-inclusive range,
  s = fp16 round-up of (hi - lo) / (2^b - 1) floored at 2^-14, z = rint(-lo / s),
  q = clip(rint(w / s) + z, 0, 2^b - 1); constant groups c get s = |c| (1 if c == 0) and
  z = 1 if c < 0 else 0.
* ``dequant`` -- Eq. (1): w_hat = s * (q - z).
* ``pack`` / ``unpack`` -- the packed record layout, from its field table (see ``_field_table``).
* ``gemm`` -- numpy.matmul in float64 of X and W_hat.
"""
import numpy as np

GROUP = 128
_MIN_NORMAL16 = np.float16(2.0 ** -14)


def quantize_rtn(W, bits):
    W = np.asarray(W, np.float16)
    K, N = W.shape
    assert K % GROUP == 0
    qmax = (1 << bits) - 1
    G = K // GROUP
    w = W.astype(np.float64).reshape(G, GROUP, N)
    lo = w.min(axis=1)
    hi = w.max(axis=1)
    const = lo == hi
    lo0 = np.minimum(lo, 0.0)
    hi0 = np.maximum(hi, 0.0)
    with np.errstate(divide="ignore", invalid="ignore"):
        sd = (hi0 - lo0) / qmax
        s16 = sd.astype(np.float16)                       # round to nearest ...
        up = s16.astype(np.float64) < sd                  # ... then up to the next fp16 if below
        s16 = np.where(up, np.nextafter(s16, np.float16(np.inf)), s16)
        down = np.nextafter(s16, np.float16(0)).astype(np.float64) >= sd
        s16 = np.where(down & (s16 > 0), np.nextafter(s16, np.float16(0)), s16)
        s16 = np.where(s16 < _MIN_NORMAL16, _MIN_NORMAL16, s16)
        c16 = lo.astype(np.float16)
        s16 = np.where(const, np.where(lo != 0.0, np.abs(c16), np.float16(1.0)), s16)
        sv = s16.astype(np.float64)
        z = np.where(const, (lo < 0.0).astype(np.float64), np.rint(-lo0 / sv))
        q = np.rint(w / sv[:, None, :]) + z[:, None, :]
    q = np.clip(q, 0, qmax)
    return (q.reshape(K, N).astype(np.uint8), s16.astype(np.float16), z.astype(np.uint8))


def dequant(codes, s, z):
    codes = np.asarray(codes)
    K, N = codes.shape
    G = K // GROUP
    sv = np.asarray(s, np.float16).astype(np.float64)
    zv = np.asarray(z).astype(np.float64)
    q = codes.astype(np.float64).reshape(G, GROUP, N)
    return (sv[:, None, :] * (q - zv[:, None, :])).reshape(K, N)


def gemm(X, codes, s, z):
    X = np.asarray(X, np.float16).astype(np.float64)
    return X @ dequant(codes, s, z)


def _field_table(bits):
    """Arrays over (lane, word, bit) of the row-in-group kk, column-in-tile nn and code bit cb,
    and the word offset of (lane, word) in the record.

    Lane l: c = l % 4, r = l / 4.  Pair (j, h, row) = codes at rows 32c + 4j + 2h + e of the group
    (e = 0 in bits 0..15, e = 1 in bits 16..31) of column r (row 0) or r + 8 (row 1).
      b = 4: word j; half-bit fields of 4 bits: (h=0,row0), (h=1,row0), (h=0,row1), (h=1,row1).
      b = 3: pair i = 2j + h; half-bit 0 carries bit w%3 of pair (15, row 0 if w < 3 else
             row 1); fields of 3 bits at half-bits 1, 4, 7, 10, 13 carry pairs (w,row0),
             (6+w,row0), (12+w//2,row w%2), (w,row1), (6+w,row1).
    """
    wpl = 8 if bits == 4 else 6
    L, Wd, B = np.meshgrid(np.arange(32), np.arange(wpl), np.arange(32), indexing="ij")
    c, r = L % 4, L // 4
    e, hb = B // 16, B % 16
    if bits == 4:
        f = hb // 4
        cb = hb % 4
        j, h, row = Wd, f % 2, f // 2
    else:
        spare = hb == 0
        field = np.where(spare, 0, (hb - 1) // 3)          # 0..4 for half-bits 1..15
        i = np.select([spare, field == 0, field == 1, field == 2, field == 3],
                      [15 + 0 * Wd, Wd, 6 + Wd, 12 + Wd // 2, Wd], 6 + Wd)
        row = np.select([spare, field == 0, field == 1, field == 2, field == 3],
                        [(Wd >= 3).astype(int), 0 * Wd, 0 * Wd, Wd % 2, 0 * Wd + 1], 0 * Wd + 1)
        cb = np.where(spare, Wd % 3, hb - 1 - 3 * field)
        j, h = i // 2, i % 2
    kk = 32 * c + 4 * j + 2 * h + e
    nn = r + 8 * row
    lw_l, lw_w = np.meshgrid(np.arange(32), np.arange(wpl), indexing="ij")
    if bits == 4:
        off = (lw_w // 4) * 128 + 4 * lw_l + lw_w % 4
    else:
        off = np.where(lw_w < 4, 4 * lw_l + lw_w, 128 + 2 * lw_l + (lw_w - 4))
    return kk, nn, cb, off


def pack(codes, bits):
    codes = np.asarray(codes, np.uint8)
    K, N = codes.shape
    assert K % GROUP == 0 and N % 16 == 0
    G, T = K // GROUP, N // 16
    kk, nn, cb, off = _field_table(bits)
    # tiles[t, g, kk, nn] = codes[128 g + kk, 16 t + nn]
    tiles = codes.reshape(G, GROUP, T, 16).transpose(2, 0, 1, 3)
    bitv = (tiles[:, :, kk, nn] >> cb.astype(np.uint8)) & 1          # [T, G, 32, wpl, 32]
    words = (bitv.astype(np.uint64) << np.arange(32, dtype=np.uint64)).sum(axis=-1)
    rec_words = 32 * (8 if bits == 4 else 6)
    out = np.zeros((T, G, rec_words), np.uint32)
    out[:, :, off] = words.astype(np.uint32)
    return out.reshape(-1)


def unpack(packed, K, N, bits):
    G, T = K // GROUP, N // 16
    kk, nn, cb, off = _field_table(bits)
    rec_words = 32 * (8 if bits == 4 else 6)
    recs = np.asarray(packed, np.uint32).reshape(T, G, rec_words)
    words = recs[:, :, off]                                            # [T, G, 32, wpl]
    bitv = (words[..., None] >> np.arange(32, dtype=np.uint32)) & 1    # [T, G, 32, wpl, 32]
    tiles = np.zeros((T, G, GROUP, 16), np.uint8)
    contrib = (bitv << cb.astype(np.uint32)).astype(np.uint8)
    np.add.at(tiles, (slice(None), slice(None), kk, nn), contrib)
    return tiles.transpose(1, 2, 0, 3).reshape(K, N)
