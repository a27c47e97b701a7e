"""The decode-step weight pass: every quantized projection of a Qwen3-shaped decoder, once.

One decode step of a batch-1 (or batch-M) decoder multiplies the current activations by each of
the 7 projections (q, k, v, o, gate, up, down) of each of the 36 layers (Sec. 5.2, "Inference":
decoding speed is bounded by streaming these weights).  ``WeightPass`` quantizes synthetic
weights with ``laq_quantize_rtn``, packs them with ``laq_pack``, and launches the 252
``laq_gemm_wxg128`` calls in stream order, optionally captured into one CUDA graph.  The
activations and outputs are per-projection slices of two flat buffers, so one host-to-device
copy feeds a whole step and one device-to-host copy returns it (the attention, norms and SiLU
between the projections are outside this pass).
"""
import torch

from . import _lib, inputs


class QuantLinear:
    """One projection's packed codes, scales and zeros on the device."""

    def __init__(self, W, bits):
        K, N = W.shape
        codes, s, z = _lib.laq_quantize_rtn(W, bits)
        self.packed = _lib.laq_pack(codes, bits)
        self.s, self.z = s, z
        self.K, self.N, self.bits = K, N, bits
        del codes

    def bytes_per_call(self, M):
        """Algorithmic HBM bytes of one call: packed codes + s (2 B) + z (1 B) per (group,
        column) + X + Y."""
        return (self.K * self.N * self.bits // 8 + (self.K // 128) * self.N * 3
                + 2 * M * self.K + 2 * M * self.N)


def shapes(model):
    return {"qwen3-4b": inputs.QWEN3_4B, "qwen3-8b": inputs.QWEN3_8B}[model]


class WeightPass:
    def __init__(self, model="qwen3-4b", bits=3, M=1, layers=inputs.LAYERS, seed=0,
                 outliers=False, device="cuda"):
        self.model, self.bits, self.M, self.layers = model, bits, M, layers
        self.seed, self.outliers = seed, outliers
        self.device = torch.device(device)
        self.linears = []   # [(layer, proj_index, name, QuantLinear)]
        plan = [(layer, pi, name, K, N) for layer in range(layers)
                for pi, (name, K, N) in enumerate(shapes(model))]
        xs = sum(M * K for *_, K, N in plan)
        ys = sum(M * N for *_, K, N in plan)
        self.Xbuf = torch.empty((xs,), dtype=torch.float16, device=self.device)
        self.Ybuf = torch.zeros((ys,), dtype=torch.float16, device=self.device)
        self.X, self.Y = [], []
        xo = yo = 0
        for layer, pi, name, K, N in plan:
            sd = inputs.proj_seed(seed, layer, pi)
            W = self.weight(layer, pi)
            self.linears.append((layer, pi, name, QuantLinear(W, bits)))
            del W
            x = self.Xbuf[xo:xo + M * K].view(M, K)
            x.copy_(inputs.activations_torch(M, K, sd, self.device))
            self.X.append(x)
            self.Y.append(self.Ybuf[yo:yo + M * N].view(M, N))
            xo += M * K
            yo += M * N
        self.configs = [None] * len(self.linears)
        torch.cuda.synchronize(self.device)

    def weight(self, layer, proj_index):
        """The fp16 weight of one projection, regenerated from its seed."""
        _, K, N = shapes(self.model)[proj_index]
        return inputs.weights_torch(K, N, inputs.proj_seed(self.seed, layer, proj_index),
                                    self.device, outliers=self.outliers)

    @property
    def launches(self):
        return len(self.linears)

    def bytes_per_pass(self):
        return sum(q.bytes_per_call(self.M) for *_, q in self.linears)

    def set_configs(self, configs):
        self.configs = list(configs)

    def run(self, stream=None, events=None):
        """Launch the pass; with ``events`` (launches + 1 CUDA events) record one before each
        launch and one after the last."""
        for i, (*_, q) in enumerate(self.linears):
            if events is not None:
                events[i].record(stream)
            _lib.laq_gemm_wxg128(self.X[i], q.packed, q.s, q.z, q.bits, Y=self.Y[i],
                                 config=self.configs[i], stream=stream)
        if events is not None:
            events[-1].record(stream)

    def capture(self, stream=None, events=None):
        """Warm every variant up (first calls set kernel attributes), then capture the pass
        into one CUDA graph and return it.  ``events`` must be created with external=True to
        become timing nodes of the graph."""
        self.run()
        torch.cuda.synchronize(self.device)
        g = torch.cuda.CUDAGraph()
        s = torch.cuda.Stream(self.device) if stream is None else stream
        with torch.cuda.graph(g, stream=s):
            self.run(stream=s, events=events)
        return g
