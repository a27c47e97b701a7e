"""ctypes binding of liblaq.so (include/laq.h): argument marshalling only.

Every function here forwards to the C entry point of the same name; all work runs in the
library's CUDA kernels.  Tensors must live on the current CUDA device; work is enqueued on the
current torch stream unless ``stream`` is given.  There is no CPU fallback: if the library is
missing or cannot be loaded, ``lib()`` raises.
"""
import ctypes
import functools
import os

PKG = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(PKG, "liblaq.so")

STATUS = {0: "LAQ_OK", 1: "LAQ_ERR_NULL", 2: "LAQ_ERR_BITS", 3: "LAQ_ERR_GROUP",
          4: "LAQ_ERR_SHAPE", 5: "LAQ_ERR_ALIGN", 6: "LAQ_ERR_M_RANGE", 7: "LAQ_ERR_CUDA",
          8: "LAQ_ERR_TIMEOUT", 9: "LAQ_ERR_CONFIG", 10: "LAQ_ERR_WORKSPACE"}

# Symbols include/laq.h declares.
EXPORTS = ("laq_status_str", "laq_version", "laq_packed_bytes", "laq_quantize_rtn", "laq_pack",
           "laq_unpack", "laq_gemm_wxg128", "laq_gemm_plan", "laq_gemm_wxg128_config",
           "laq_chain_workspace_bytes", "laq_gemm_chain", "laq_gemm_chain_static")
CHAIN_MAX = 384  # LAQ_CHAIN_MAX


class LaqError(RuntimeError):
    def __init__(self, status, where):
        self.status = status
        super().__init__(f"{where}: {lib().laq_status_str(status).decode()} (status {status})")


class GemmConfig(ctypes.Structure):
    _fields_ = [("tiles_per_cta", ctypes.c_int32), ("warps", ctypes.c_int32),
                ("cluster", ctypes.c_int32), ("stages", ctypes.c_int32), ("pdl", ctypes.c_int32),
                ("reserved", ctypes.c_int32 * 3)]

    def as_dict(self):
        return {"tiles_per_cta": self.tiles_per_cta, "warps": self.warps,
                "cluster": self.cluster, "stages": self.stages, "pdl": self.pdl}

    @classmethod
    def make(cls, tiles_per_cta, warps, cluster, stages, pdl=0):
        return cls(tiles_per_cta, warps, cluster, stages, pdl, (ctypes.c_int32 * 3)(0, 0, 0))


class Gemv(ctypes.Structure):
    """struct laq_gemv: one entry of a laq_gemm_chain call."""
    _fields_ = [("X", ctypes.c_void_p), ("packed", ctypes.c_void_p), ("s", ctypes.c_void_p),
                ("z", ctypes.c_void_p), ("Y", ctypes.c_void_p), ("M", ctypes.c_int64),
                ("K", ctypes.c_int64), ("N", ctypes.c_int64), ("bits", ctypes.c_int32),
                ("wait_prev", ctypes.c_int32)]


@functools.lru_cache(maxsize=1)
def lib():
    if not os.path.exists(LIB_PATH):
        raise RuntimeError(f"{LIB_PATH} is missing: build it with "
                           "`python -c 'import __graft_entry__ as g; g.build()'`")
    L = ctypes.CDLL(LIB_PATH)
    P, I64, I = ctypes.c_void_p, ctypes.c_int64, ctypes.c_int
    L.laq_status_str.argtypes = [I]
    L.laq_status_str.restype = ctypes.c_char_p
    L.laq_version.argtypes = []
    L.laq_version.restype = I
    L.laq_packed_bytes.argtypes = [I64, I64, I]
    L.laq_packed_bytes.restype = ctypes.c_size_t
    L.laq_quantize_rtn.argtypes = [P, I64, I64, I, I, P, P, P, P]
    L.laq_pack.argtypes = [P, I64, I64, I, P, P]
    L.laq_unpack.argtypes = [P, I64, I64, I, P, P]
    L.laq_gemm_wxg128.argtypes = [P, I64, I64, I64, P, P, P, I, P, P]
    L.laq_gemm_plan.argtypes = [I64, I64, I64, I, I, ctypes.POINTER(GemmConfig)]
    L.laq_gemm_wxg128_config.argtypes = [P, I64, I64, I64, P, P, P, I, P,
                                         ctypes.POINTER(GemmConfig), P]
    L.laq_chain_workspace_bytes.argtypes = [ctypes.c_int32]
    L.laq_chain_workspace_bytes.restype = ctypes.c_size_t
    L.laq_gemm_chain.argtypes = [ctypes.POINTER(Gemv), ctypes.c_int32, P, ctypes.c_size_t, P]
    L.laq_gemm_chain_static.argtypes = [ctypes.POINTER(Gemv), ctypes.c_int32, P]
    for name in ("laq_quantize_rtn", "laq_pack", "laq_unpack", "laq_gemm_wxg128",
                 "laq_gemm_plan", "laq_gemm_wxg128_config", "laq_gemm_chain",
                 "laq_gemm_chain_static"):
        getattr(L, name).restype = I
    return L


def _check(status, where):
    if status != 0:
        raise LaqError(status, where)


def _ptr(t):
    return None if t is None else ctypes.c_void_p(t.data_ptr())


def _stream(stream):
    import torch
    s = torch.cuda.current_stream() if stream is None else stream
    return ctypes.c_void_p(s.cuda_stream)


def packed_bytes(K, N, bits):
    return int(lib().laq_packed_bytes(K, N, bits))


def laq_quantize_rtn(W, bits, group=128, stream=None):
    """W [K, N] fp16 (CUDA) -> (codes u8 [K, N], s fp16 [K/128, N], z u8 [K/128, N])."""
    import torch
    K, N = W.shape
    G = K // 128
    codes = torch.empty((K, N), dtype=torch.uint8, device=W.device)
    s = torch.empty((G, N), dtype=torch.float16, device=W.device)
    z = torch.empty((G, N), dtype=torch.uint8, device=W.device)
    W = W.contiguous()
    _check(lib().laq_quantize_rtn(_ptr(W), K, N, bits, group, _ptr(codes), _ptr(s), _ptr(z),
                                  _stream(stream)), "laq_quantize_rtn")
    return codes, s, z


def laq_pack(codes, bits, stream=None):
    """codes u8 [K, N] (CUDA) -> packed uint8 [K * N * bits / 8] in the library's layout."""
    import torch
    K, N = codes.shape
    packed = torch.empty((K * N * bits // 8,), dtype=torch.uint8, device=codes.device)
    codes = codes.contiguous()
    _check(lib().laq_pack(_ptr(codes), K, N, bits, _ptr(packed), _stream(stream)), "laq_pack")
    return packed


def laq_unpack(packed, K, N, bits, stream=None):
    import torch
    codes = torch.empty((K, N), dtype=torch.uint8, device=packed.device)
    _check(lib().laq_unpack(_ptr(packed), K, N, bits, _ptr(codes), _stream(stream)),
           "laq_unpack")
    return codes


def laq_gemm_wxg128(X, packed, s, z, bits, Y=None, config=None, stream=None):
    """Y[M, N] = X[M, K] * W_hat[K, N] (fp16 in/out).  ``config``: optional GemmConfig."""
    import torch
    M, K = X.shape
    N = s.shape[1]
    if Y is None:
        Y = torch.empty((M, N), dtype=torch.float16, device=X.device)
    args = (_ptr(X), M, K, N, _ptr(packed), _ptr(s), _ptr(z), bits, _ptr(Y))
    if config is None:
        _check(lib().laq_gemm_wxg128(*args, _stream(stream)), "laq_gemm_wxg128")
    else:
        _check(lib().laq_gemm_wxg128_config(*args, ctypes.byref(config), _stream(stream)),
               "laq_gemm_wxg128_config")
    return Y


def laq_gemm_plan(M, K, N, bits, num_sms):
    cfg = GemmConfig()
    _check(lib().laq_gemm_plan(M, K, N, bits, num_sms, ctypes.byref(cfg)), "laq_gemm_plan")
    return cfg


def laq_chain_workspace_bytes(count):
    return int(lib().laq_chain_workspace_bytes(count))


def chain_workspace(count, device):
    """A zero-filled workspace for chains of up to ``count`` entries."""
    import torch
    n = laq_chain_workspace_bytes(count)
    if n == 0:
        raise ValueError(f"chain length {count} outside 0..{CHAIN_MAX}")
    return torch.zeros((n,), dtype=torch.uint8, device=device)


class Chain:
    """A fixed list of GEMVs for laq_gemm_chain: entries are (X, packed, s, z, bits, Y,
    wait_prev) with device tensors, kept alive here so the call can be replayed (or captured)."""

    def __init__(self, entries):
        self.tensors = []
        self.array = (Gemv * max(1, len(entries)))()
        for i, (X, packed, s, z, bits, Y, wait_prev) in enumerate(entries):
            M, K = X.shape
            N = s.shape[1]
            self.array[i] = Gemv(X.data_ptr(), packed.data_ptr(), s.data_ptr(), z.data_ptr(),
                                 Y.data_ptr(), M, K, N, bits, 1 if wait_prev else 0)
            self.tensors.append((X, packed, s, z, Y))
        self.count = len(entries)

    def run(self, workspace, stream=None):
        ws = workspace
        _check(lib().laq_gemm_chain(self.array, self.count, _ptr(ws), ws.numel(),
                                    _stream(stream)), "laq_gemm_chain")

    def run_static(self, stream=None):
        """The same chain through laq_gemm_chain_static (the library's own scratch)."""
        _check(lib().laq_gemm_chain_static(self.array, self.count, _stream(stream)),
               "laq_gemm_chain_static")


def laq_gemm_chain(entries, workspace, stream=None):
    """Run ``entries`` (see ``Chain``) as one persistent launch on ``stream``."""
    Chain(entries).run(workspace, stream)


def chain_status(workspace):
    """The device-side status word of a chain workspace (synchronizes the device)."""
    import torch
    torch.cuda.synchronize(workspace.device)
    return int(workspace[:4].view(torch.int32)[0].item())
