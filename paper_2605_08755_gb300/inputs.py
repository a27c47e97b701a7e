"""Seeded synthetic inputs shared by the tests, the benchmark and the smoke check.

This module only draws random numbers and names shapes; it holds none of the quantizer's or the
GEMV's arithmetic.  The synthetic tensors stand in for the weights and activations of the
Qwen3-4B / Qwen3-8B decoders quantized in the paper (their checkpoints and calibration data are
not used):

* weights  W[K, N] fp16 ~ N(0, 0.02^2); the 8B-shaped workload multiplies an iid Bernoulli(0.01)
  mask of entries by 20 before rounding to fp16 ("1% outliers x20");
* activations X[M, K] fp16 ~ N(0, 1).

Host (numpy) generators serve small cases; the torch generators draw the same distributions on a
device for the 36-layer passes.  Seeds are derived as base + 1000 * layer + projection index, with
projections in the order q, k, v, o, gate, up, down.
"""
import numpy as np

# (name, K = in_features, N = out_features) of one decoder layer, W stored [K, N].
QWEN3_4B = (("q", 2560, 4096), ("k", 2560, 1024), ("v", 2560, 1024), ("o", 4096, 2560),
            ("gate", 2560, 9728), ("up", 2560, 9728), ("down", 9728, 2560))
QWEN3_8B = (("q", 4096, 4096), ("k", 4096, 1024), ("v", 4096, 1024), ("o", 4096, 4096),
            ("gate", 4096, 12288), ("up", 4096, 12288), ("down", 12288, 4096))
LAYERS = 36
W_STD = 0.02
OUTLIER_FRAC = 0.01
OUTLIER_SCALE = 20.0


def proj_seed(base: int, layer: int, proj_index: int) -> int:
    return base + 1000 * layer + proj_index


def weights(K, N, seed, outliers=False):
    rng = np.random.default_rng(seed)
    w = rng.standard_normal((K, N), dtype=np.float32) * np.float32(W_STD)
    if outliers:
        mask = rng.random((K, N), dtype=np.float32) < OUTLIER_FRAC
        w = np.where(mask, w * np.float32(OUTLIER_SCALE), w)
    return w.astype(np.float16)


def activations(M, K, seed):
    rng = np.random.default_rng(seed + 7_777_777)
    return rng.standard_normal((M, K), dtype=np.float32).astype(np.float16)


def weights_torch(K, N, seed, device, outliers=False):
    import torch
    g = torch.Generator(device=device)
    g.manual_seed(seed)
    w = torch.randn((K, N), generator=g, device=device, dtype=torch.float32) * W_STD
    if outliers:
        mask = torch.rand((K, N), generator=g, device=device) < OUTLIER_FRAC
        w = torch.where(mask, w * OUTLIER_SCALE, w)
    return w.to(torch.float16)


def activations_torch(M, K, seed, device):
    import torch
    g = torch.Generator(device=device)
    g.manual_seed(seed + 7_777_777)
    return torch.randn((M, K), generator=g, device=device, dtype=torch.float32).to(torch.float16)


# ---- the rest of a decode step (synthetic stand-ins; no checkpoint is used) ----

# Decoder dimensions of the two Qwen3 models (their public configurations): hidden size H,
# q heads, kv heads, head size D, MLP width I, vocabulary V, rotary base, RMSNorm epsilon.
DECODER = {
    "qwen3-4b": dict(H=2560, Hq=32, Hkv=8, D=128, I=9728, V=151936, theta=1e6, eps=1e-6),
    "qwen3-8b": dict(H=4096, Hq=32, Hkv=8, D=128, I=12288, V=151936, theta=1e6, eps=1e-6),
}
NORM_STD = 0.1      # norm weights ~ 1 + N(0, 0.1^2)
EMBED_STD = 0.05    # embedding rows ~ N(0, 0.05^2)


def norm_weight(n, seed):
    rng = np.random.default_rng(seed + 5_555_555)
    return (1.0 + NORM_STD * rng.standard_normal(n, dtype=np.float32)).astype(np.float16)


def embedding(V, H, seed):
    rng = np.random.default_rng(seed + 3_333_333)
    return (EMBED_STD * rng.standard_normal((V, H), dtype=np.float32)).astype(np.float16)


def kv_cache(M, Hkv, L, D, seed):
    """Cached keys or values ~ N(0, 1) for the tokens before the new one."""
    rng = np.random.default_rng(seed + 1_111_111)
    return rng.standard_normal((M, Hkv, L, D), dtype=np.float32).astype(np.float16)


def tokens(M, V, seed):
    rng = np.random.default_rng(seed + 9_999_999)
    return rng.integers(0, V, size=M).astype(np.int32)


def norm_weight_torch(n, seed, device):
    import torch
    g = torch.Generator(device=device)
    g.manual_seed(seed + 5_555_555)
    return (1.0 + NORM_STD * torch.randn(n, generator=g, device=device)).to(torch.float16)


def embedding_torch(V, H, seed, device):
    import torch
    g = torch.Generator(device=device)
    g.manual_seed(seed + 3_333_333)
    return (EMBED_STD * torch.randn((V, H), generator=g, device=device)).to(torch.float16)


def kv_cache_torch(M, Hkv, L, D, seed, device):
    import torch
    g = torch.Generator(device=device)
    g.manual_seed(seed + 1_111_111)
    return torch.randn((M, Hkv, L, D), generator=g, device=device).to(torch.float16)


# ---- the online pairwise rotation of a projection's input (the rotation-based comparison) ----

def rotation(K, rounds, seed):
    """Tables of a pairwise rotation of K channels: per 128-channel group and round, a random
    perfect matching of the group's channels into 64 pairs (uint8 [K/128][rounds][64][2]), one
    angle per pair (float32 [K/128][rounds][64], uniform in [-pi, pi)), and channel scales
    (fp16 [K], 1 + N(0, 0.1^2))."""
    rng = np.random.default_rng(seed + 4_444_444)
    G = K // 128
    pairs = np.stack([rng.permutation(128).astype(np.uint8).reshape(64, 2)
                      for _ in range(G * rounds)]).reshape(G, rounds, 64, 2)
    theta = rng.uniform(-np.pi, np.pi, size=(G, rounds, 64)).astype(np.float32)
    alpha = (1.0 + NORM_STD * rng.standard_normal(K, dtype=np.float32)).astype(np.float16)
    return pairs, theta, alpha
