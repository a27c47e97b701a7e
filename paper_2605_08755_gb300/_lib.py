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
           "laq_chain_workspace_bytes", "laq_gemm_chain", "laq_gemm_chain_static",
           "laq_gemm_wxg128_prologue",
           "laq_rmsnorm", "laq_qk_norm_rope", "laq_attention_workspace_bytes",
           "laq_attention_decode", "laq_attention_qkv_workspace_bytes", "laq_attention_qkv",
           "laq_silu_mul", "laq_embed", "laq_argmax", "laq_rotation_tables",
           "laq_pairwise_rotate", "laq_pass_plan_sizes", "laq_pass_plan_build",
           "laq_pass_workspace_bytes", "laq_pass_prepare", "laq_pass_run")
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


class GemmPrologue(ctypes.Structure):
    """struct laq_gemm_prologue."""
    _fields_ = [("kind", ctypes.c_int32), ("eps", ctypes.c_float), ("R", ctypes.c_void_p),
                ("R_out", ctypes.c_void_p), ("w", ctypes.c_void_p)]


PROLOGUE_NONE, PROLOGUE_RMSNORM, PROLOGUE_SILU_MUL = 0, 1, 2


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
    L.laq_gemm_wxg128_prologue.argtypes = [P, I64, I64, I64, P, P, P, I, P,
                                           ctypes.POINTER(GemmPrologue),
                                           ctypes.POINTER(GemmConfig), P]
    L.laq_chain_workspace_bytes.argtypes = [ctypes.c_int32]
    L.laq_chain_workspace_bytes.restype = ctypes.c_size_t
    L.laq_gemm_chain.argtypes = [ctypes.POINTER(Gemv), ctypes.c_int32, P, ctypes.c_size_t, P]
    L.laq_gemm_chain_static.argtypes = [ctypes.POINTER(Gemv), ctypes.c_int32, P]
    F, I32, SZ = ctypes.c_float, ctypes.c_int32, ctypes.c_size_t
    L.laq_rmsnorm.argtypes = [P, P, P, P, I64, I64, F, P, P]
    L.laq_qk_norm_rope.argtypes = [P, P, P, P, I64, I32, I32, I32, F, F, P, P, P, I64, P]
    L.laq_attention_workspace_bytes.argtypes = [I64, I32, I64]
    L.laq_attention_workspace_bytes.restype = SZ
    L.laq_attention_decode.argtypes = [P, P, P, P, I64, I32, I32, I32, I64, F, P, P, SZ, P]
    L.laq_attention_qkv_workspace_bytes.argtypes = [I64, I32, I32, I64]
    L.laq_attention_qkv_workspace_bytes.restype = SZ
    L.laq_attention_qkv.argtypes = [P, P, P, P, I64, I32, I32, I32, F, F, P, P, I64, F, P, P, SZ,
                                    P]
    L.laq_silu_mul.argtypes = [P, I64, I64, P, P]
    L.laq_embed.argtypes = [P, P, I64, I64, I64, P, P]
    L.laq_argmax.argtypes = [P, I64, I64, P, P]
    L.laq_rotation_tables.argtypes = [P, I64, P, P]
    L.laq_pairwise_rotate.argtypes = [P, I64, I64, P, P, P, I32, P, P]
    L.laq_pass_plan_sizes.argtypes = [ctypes.POINTER(Gemv), I32, I32, ctypes.POINTER(SZ),
                                      ctypes.POINTER(SZ)]
    L.laq_pass_plan_build.argtypes = [ctypes.POINTER(Gemv), I32, I32, P, SZ]
    L.laq_pass_workspace_bytes.argtypes = [P]
    L.laq_pass_workspace_bytes.restype = SZ
    L.laq_pass_prepare.argtypes = [P, P, SZ, P]
    L.laq_pass_run.argtypes = [P, P, P, SZ, P]
    for name in ("laq_quantize_rtn", "laq_pack", "laq_unpack", "laq_gemm_wxg128",
                 "laq_gemm_plan", "laq_gemm_wxg128_config", "laq_gemm_chain",
                 "laq_gemm_chain_static", "laq_rmsnorm", "laq_qk_norm_rope",
                 "laq_gemm_wxg128_prologue",
                 "laq_attention_decode", "laq_attention_qkv", "laq_silu_mul", "laq_embed",
                 "laq_argmax", "laq_rotation_tables", "laq_pairwise_rotate",
                 "laq_pass_plan_sizes", "laq_pass_plan_build", "laq_pass_prepare",
                 "laq_pass_run"):
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


def laq_gemm_wxg128_prologue(X, packed, s, z, bits, kind, Y=None, R=None, R_out=None, w=None,
                             eps=0.0, config=None, stream=None):
    """laq_gemm_wxg128 whose input is a prologue of X: PROLOGUE_RMSNORM (rmsnorm(X + R) * w,
    R_out = fp16(X + R)) or PROLOGUE_SILU_MUL (X [M, 2K] = gate | up -> silu(gate) * up)."""
    import torch
    M = X.shape[0]
    K = X.shape[1] // 2 if kind == PROLOGUE_SILU_MUL else X.shape[1]
    N = s.shape[1]
    if Y is None:
        Y = torch.empty((M, N), dtype=torch.float16, device=X.device)
    pro = GemmPrologue(kind, float(eps), None if R is None else R.data_ptr(),
                       None if R_out is None else R_out.data_ptr(),
                       None if w is None else w.data_ptr())
    _check(lib().laq_gemm_wxg128_prologue(_ptr(X), M, K, N, _ptr(packed), _ptr(s), _ptr(z), bits,
                                          _ptr(Y), ctypes.byref(pro),
                                          None if config is None else ctypes.byref(config),
                                          _stream(stream)), "laq_gemm_wxg128_prologue")
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


def pass_plan(gemvs, count, num_sms):
    """Host work only: the laq_pass plan of ``count`` laq_gemv entries (a ctypes Gemv array) for
    ``num_sms`` SMs, as a ctypes byte buffer, and the device bytes it needs."""
    pb, db = ctypes.c_size_t(0), ctypes.c_size_t(0)
    _check(lib().laq_pass_plan_sizes(gemvs, count, num_sms, ctypes.byref(pb), ctypes.byref(db)),
           "laq_pass_plan_sizes")
    plan = (ctypes.c_uint8 * pb.value)()
    _check(lib().laq_pass_plan_build(gemvs, count, num_sms, plan, pb.value),
           "laq_pass_plan_build")
    return plan, db.value


class PassPlan:
    """The entries of a ``Chain`` planned for laq_pass_run on ``device``: the host plan, the
    prepared device buffer (per-SM weight streams and tables) and a zeroed workspace.  The
    entries' X and Y tensors are kept alive; their packed weights are no longer read once
    ``prepare`` has run on the stream.  laq_pass_prepare and laq_pass_run work on the current
    device, so both calls are made with ``device`` current (and, without ``stream``, on that
    device's current stream)."""

    def __init__(self, entries, device, stream=None):
        import torch
        self.chain = Chain(entries)
        self.device = torch.device(device)
        if self.device.index is None:
            self.device = torch.device("cuda", torch.cuda.current_device())
        sms = torch.cuda.get_device_properties(self.device).multi_processor_count
        self.plan, dev_bytes = pass_plan(self.chain.array, self.chain.count, sms)
        self.buffer = torch.empty((max(dev_bytes, 256),), dtype=torch.uint8, device=self.device)
        self.ws = torch.zeros((max(256, int(lib().laq_pass_workspace_bytes(self.plan))),),
                              dtype=torch.uint8, device=self.device)
        with torch.cuda.device(self.device):
            st = stream if stream is not None else torch.cuda.current_stream(self.device)
            _check(lib().laq_pass_prepare(self.plan, _ptr(self.buffer), self.buffer.numel(),
                                          _stream(st)), "laq_pass_prepare")

    def run(self, stream=None):
        import torch
        with torch.cuda.device(self.device):
            st = stream if stream is not None else torch.cuda.current_stream(self.device)
            _check(lib().laq_pass_run(self.plan, _ptr(self.buffer), _ptr(self.ws),
                                      self.ws.numel(), _stream(st)), "laq_pass_run")

    def status(self):
        """The device-side status word (synchronizes the device)."""
        return chain_status(self.ws)


# ---- decoder operations around the projections (one decode step) ----

def laq_rmsnorm(X, w, eps, R=None, R_out=None, Y=None, stream=None):
    """Y = rmsnorm(X + R) * w per row (fp16 [M, H]); with R_out, also R_out = fp16(X + R)."""
    import torch
    M, H = X.shape
    if Y is None:
        Y = torch.empty_like(X)
    _check(lib().laq_rmsnorm(_ptr(X), _ptr(R), _ptr(R_out), _ptr(w), M, H, float(eps), _ptr(Y),
                             _stream(stream)), "laq_rmsnorm")
    return Y


def laq_qk_norm_rope(qkv, q_norm_w, k_norm_w, pos, Hq, Hkv, theta, eps, k_cache, v_cache,
                     q_out=None, stream=None):
    """qkv [M, (Hq + 2 Hkv) * 128] -> q_out [M, Hq, 128]; appends k, v at pos[m] to the caches
    [M, Hkv, L_max, 128]."""
    import torch
    M = qkv.shape[0]
    D = k_cache.shape[-1]
    L_max = k_cache.shape[-2]
    if q_out is None:
        q_out = torch.empty((M, Hq, D), dtype=torch.float16, device=qkv.device)
    _check(lib().laq_qk_norm_rope(_ptr(qkv), _ptr(q_norm_w), _ptr(k_norm_w), _ptr(pos), M, Hq,
                                  Hkv, D, float(theta), float(eps), _ptr(q_out), _ptr(k_cache),
                                  _ptr(v_cache), L_max, _stream(stream)), "laq_qk_norm_rope")
    return q_out


def attention_workspace(M, Hq, L_max, device):
    import torch
    n = int(lib().laq_attention_workspace_bytes(M, Hq, L_max))
    if n == 0:
        raise ValueError("invalid attention sizes")
    return torch.empty((n // 4,), dtype=torch.float32, device=device)


def laq_attention_decode(q, k_cache, v_cache, lens, scale, workspace, out=None, stream=None):
    """out [M, Hq, 128] = GQA softmax attention of q [M, Hq, 128] over the first lens[m]
    tokens of the caches [M, Hkv, L_max, 128]."""
    import torch
    M, Hq, D = q.shape
    Hkv, L_max = k_cache.shape[1], k_cache.shape[2]
    if out is None:
        out = torch.empty_like(q)
    _check(lib().laq_attention_decode(_ptr(q), _ptr(k_cache), _ptr(v_cache), _ptr(lens), M, Hq,
                                      Hkv, D, L_max, float(scale), _ptr(out), _ptr(workspace),
                                      workspace.numel() * workspace.element_size(),
                                      _stream(stream)), "laq_attention_decode")
    return out


def attention_qkv_workspace(M, Hq, Hkv, L_max, device):
    """A workspace for laq_attention_qkv."""
    import torch
    n = int(lib().laq_attention_qkv_workspace_bytes(M, Hq, Hkv, L_max))
    if n == 0:
        raise ValueError("invalid attention sizes")
    return torch.zeros((n,), dtype=torch.uint8, device=device)


def laq_attention_qkv(qkv, q_norm_w, k_norm_w, pos, Hq, Hkv, theta, eps, k_cache, v_cache,
                      scale, workspace, out=None, stream=None):
    """laq_qk_norm_rope + laq_attention_decode (len = pos + 1) in two launches: out [M, Hq, 128];
    appends k, v at pos[m] to the caches [M, Hkv, L_max, 128]."""
    import torch
    M = qkv.shape[0]
    D, L_max = k_cache.shape[-1], k_cache.shape[-2]
    if out is None:
        out = torch.empty((M, Hq, D), dtype=torch.float16, device=qkv.device)
    _check(lib().laq_attention_qkv(_ptr(qkv), _ptr(q_norm_w), _ptr(k_norm_w), _ptr(pos), M, Hq,
                                   Hkv, D, float(theta), float(eps), _ptr(k_cache),
                                   _ptr(v_cache), L_max, float(scale), _ptr(out),
                                   _ptr(workspace), workspace.numel() * workspace.element_size(),
                                   _stream(stream)), "laq_attention_qkv")
    return out


def laq_silu_mul(gate_up, h=None, stream=None):
    """h [M, I] = silu(gate_up[:, :I]) * gate_up[:, I:]."""
    import torch
    M, I2 = gate_up.shape
    if h is None:
        h = torch.empty((M, I2 // 2), dtype=torch.float16, device=gate_up.device)
    _check(lib().laq_silu_mul(_ptr(gate_up), M, I2 // 2, _ptr(h), _stream(stream)),
           "laq_silu_mul")
    return h


def laq_embed(E, tokens, X=None, stream=None):
    """X [M, H] = E[tokens] (zero rows for tokens outside the table)."""
    import torch
    V, H = E.shape
    M = tokens.shape[0]
    if X is None:
        X = torch.empty((M, H), dtype=torch.float16, device=E.device)
    _check(lib().laq_embed(_ptr(E), _ptr(tokens), M, V, H, _ptr(X), _stream(stream)), "laq_embed")
    return X


def laq_argmax(logits, out=None, stream=None):
    """out [M] int32 = argmax over each row of fp16 logits [M, V] (ties: smallest index)."""
    import torch
    M, V = logits.shape
    if out is None:
        out = torch.empty((M,), dtype=torch.int32, device=logits.device)
    _check(lib().laq_argmax(_ptr(logits), M, V, _ptr(out), _stream(stream)), "laq_argmax")
    return out


# ---- the online pairwise rotation (the rotation-based comparison) ----

def laq_rotation_tables(theta, stream=None):
    """(cos, sin) of every angle: float32 [..., 2] for float32 angles theta [...]."""
    import torch
    cs = torch.empty(tuple(theta.shape) + (2,), dtype=torch.float32, device=theta.device)
    _check(lib().laq_rotation_tables(_ptr(theta), theta.numel(), _ptr(cs), _stream(stream)),
           "laq_rotation_tables")
    return cs


def laq_pairwise_rotate(X, pairs, cs, alpha=None, Y=None, stream=None):
    """Y [M, K] = the rotation of X: channel scales alpha [K] (or none), then the rounds of
    pairs uint8 [K/128, R, 64, 2] with (cos, sin) cs [K/128, R, 64, 2]."""
    import torch
    M, K = X.shape
    rounds = pairs.shape[1]
    if Y is None:
        Y = torch.empty((M, K), dtype=torch.float16, device=X.device)
    _check(lib().laq_pairwise_rotate(_ptr(X), M, K, _ptr(alpha), _ptr(pairs), _ptr(cs), rounds,
                                     _ptr(Y), _stream(stream)), "laq_pairwise_rotate")
    return Y
