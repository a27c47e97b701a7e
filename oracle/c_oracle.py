"""ctypes front end of the C oracle ``laq_oracle.c`` (fp64, single-threaded, slow on purpose).

TEST INFRASTRUCTURE ONLY.  Arrays are numpy; fp16 tensors travel as their uint16 bit patterns.
Each wrapper follows the C function of the same name, which cites the passage it implements
(Eq. (1) of LAQuant for the quantizer and dequantizer; the library's own packed layout).
"""
import ctypes
import functools

import numpy as np

from . import build as _build

GROUP = 128


@functools.lru_cache(maxsize=1)
def _lib():
    lib = ctypes.CDLL(_build.build())
    P = ctypes.c_void_p
    I64 = ctypes.c_int64
    I = ctypes.c_int
    sigs = {
        "laqo_quantize_rtn": [P, I64, I64, I, I, P, P, P],
        "laqo_quantize_rtn_threads": [P, I64, I64, I, I, P, P, P],
        "laqo_dequant": [P, P, P, I64, I64, P],
        "laqo_gemm": [P, I64, I64, I64, P, P, P, P],
        "laqo_gemm_columns": [P, I64, I64, I64, P, P, P, P, I64, P],
        "laqo_gemm_threads": [P, I64, I64, I64, P, P, P, P],
        "laqo_pack": [P, I64, I64, I, P],
        "laqo_unpack": [P, I64, I64, I, P],
        "laqo_layout_bit": [I, I, I, I, P, P, P],
    }
    for name, args in sigs.items():
        f = getattr(lib, name)
        f.argtypes = args
        f.restype = I
    lib.laqo_threads.argtypes = []
    lib.laqo_threads.restype = I
    lib.laqo_half_to_double.argtypes = [ctypes.c_uint16]
    lib.laqo_half_to_double.restype = ctypes.c_double
    lib.laqo_packed_words.argtypes = [I64, I64, I]
    lib.laqo_packed_words.restype = I64
    lib.laqo_word_offset.argtypes = [I, I, I]
    lib.laqo_word_offset.restype = I64
    return lib


def _ptr(a):
    return a.ctypes.data_as(ctypes.c_void_p)


def _bits16(a):
    a = np.ascontiguousarray(a)
    if a.dtype == np.float16:
        return a.view(np.uint16)
    assert a.dtype == np.uint16
    return a


def _check(rc, name):
    if rc != 0:
        raise ValueError(f"{name} returned status {rc}")


def half_to_double(bits16: int) -> float:
    return _lib().laqo_half_to_double(int(bits16))


def quantize_rtn(W, bits, group=GROUP):
    """Eq. (1) RTN min-max group quantizer.  W: [K, N] fp16.  Returns (codes u8 [K,N],
    s fp16 [K/128, N], z u8 [K/128, N])."""
    Wb = _bits16(W)
    K, N = Wb.shape
    G = K // GROUP if K % GROUP == 0 else 0
    codes = np.zeros((K, N), np.uint8)
    s = np.zeros((G, N), np.uint16)
    z = np.zeros((G, N), np.uint8)
    _check(_lib().laqo_quantize_rtn(_ptr(Wb), K, N, bits, group, _ptr(codes), _ptr(s), _ptr(z)),
           "laqo_quantize_rtn")
    return codes, s.view(np.float16), z


def quantize_rtn_threads(W, bits, group=GROUP):
    """``quantize_rtn`` with the columns split over the host's threads (bit-identical)."""
    Wb = _bits16(W)
    K, N = Wb.shape
    G = K // GROUP if K % GROUP == 0 else 0
    codes = np.zeros((K, N), np.uint8)
    s = np.zeros((G, N), np.uint16)
    z = np.zeros((G, N), np.uint8)
    _check(_lib().laqo_quantize_rtn_threads(_ptr(Wb), K, N, bits, group, _ptr(codes), _ptr(s),
                                            _ptr(z)), "laqo_quantize_rtn_threads")
    return codes, s.view(np.float16), z


def dequant(codes, s, z):
    """Eq. (1): w_hat = s * (q - z) in fp64.  Returns [K, N] float64."""
    codes = np.ascontiguousarray(codes, np.uint8)
    K, N = codes.shape
    out = np.zeros((K, N), np.float64)
    _check(_lib().laqo_dequant(_ptr(codes), _ptr(_bits16(s)), _ptr(np.ascontiguousarray(z)),
                               K, N, _ptr(out)), "laqo_dequant")
    return out


def gemm(X, codes, s, z):
    """Y = X * W_hat in fp64 (naive k-ascending sums).  X: [M, K] fp16.  Returns [M, N] f64."""
    Xb = _bits16(X)
    M, K = Xb.shape
    codes = np.ascontiguousarray(codes, np.uint8)
    N = codes.shape[1]
    Y = np.zeros((M, N), np.float64)
    _check(_lib().laqo_gemm(_ptr(Xb), M, K, N, _ptr(codes), _ptr(_bits16(s)),
                            _ptr(np.ascontiguousarray(z)), _ptr(Y)), "laqo_gemm")
    return Y


def gemm_threads(X, codes, s, z):
    """``gemm`` with the output columns split over the host's threads (bit-identical)."""
    Xb = _bits16(X)
    M, K = Xb.shape
    codes = np.ascontiguousarray(codes, np.uint8)
    N = codes.shape[1]
    Y = np.zeros((M, N), np.float64)
    _check(_lib().laqo_gemm_threads(_ptr(Xb), M, K, N, _ptr(codes), _ptr(_bits16(s)),
                                    _ptr(np.ascontiguousarray(z)), _ptr(Y)), "laqo_gemm_threads")
    return Y


def threads():
    """Threads ``gemm_threads`` runs with (OMP_NUM_THREADS, else every available core)."""
    return int(_lib().laqo_threads())


def gemm_columns(X, codes, s, z, cols):
    """Y[:, cols] of ``gemm`` computed one output at a time.  Returns [M, len(cols)] f64."""
    Xb = _bits16(X)
    M, K = Xb.shape
    codes = np.ascontiguousarray(codes, np.uint8)
    N = codes.shape[1]
    cols = np.ascontiguousarray(cols, np.int64)
    Y = np.zeros((M, len(cols)), np.float64)
    _check(_lib().laqo_gemm_columns(_ptr(Xb), M, K, N, _ptr(codes), _ptr(_bits16(s)),
                                    _ptr(np.ascontiguousarray(z)), _ptr(cols), len(cols),
                                    _ptr(Y)), "laqo_gemm_columns")
    return Y


def packed_words(K, N, bits):
    return int(_lib().laqo_packed_words(K, N, bits))


def pack(codes, bits):
    """Codes [K, N] u8 -> packed uint32 words in the library's record layout."""
    codes = np.ascontiguousarray(codes, np.uint8)
    K, N = codes.shape
    out = np.zeros(packed_words(K, N, bits), np.uint32)
    _check(_lib().laqo_pack(_ptr(codes), K, N, bits, _ptr(out)), "laqo_pack")
    return out


def unpack(packed, K, N, bits):
    packed = np.ascontiguousarray(packed, np.uint32)
    codes = np.zeros((K, N), np.uint8)
    _check(_lib().laqo_unpack(_ptr(packed), K, N, bits, _ptr(codes)), "laqo_unpack")
    return codes


def layout_bit(bits, lane, word, bit):
    """(row-in-group, column-in-tile, code bit) carried by one bit of the packed record."""
    kk, nn, cb = ctypes.c_int(), ctypes.c_int(), ctypes.c_int()
    _check(_lib().laqo_layout_bit(bits, lane, word, bit, ctypes.byref(kk), ctypes.byref(nn),
                                  ctypes.byref(cb)), "laqo_layout_bit")
    return kk.value, nn.value, cb.value


def word_offset(bits, lane, word):
    return int(_lib().laqo_word_offset(bits, lane, word))
