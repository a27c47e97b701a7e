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
