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


# Projections that read the same activation and may run as one GEMV over concatenated columns.
FUSED = (("qkv", ("q", "k", "v")), ("o", ("o",)), ("gate_up", ("gate", "up")), ("down", ("down",)))
# Projections whose input is the previous projection's input (they need nothing new).
SHARES_INPUT = {"k", "v", "up"}


def pass_plan(model, fuse, layers):
    """The pass's GEMVs in launch order: (layer, member projection indices, name, K, N)."""
    names = [n for n, _, _ in shapes(model)]
    groups = ([[names.index(m) for m in members] for _, members in FUSED] if fuse
              else [[i] for i in range(len(names))])
    gnames = [n for n, _ in FUSED] if fuse else names
    plan = []
    for layer in range(layers):
        for gname, members in zip(gnames, groups):
            K = shapes(model)[members[0]][1]
            N = sum(shapes(model)[i][2] for i in members)
            plan.append((layer, tuple(members), gname, K, N))
    return plan


class WeightPass:
    """The 7 x layers projections of a decode step, launched in stream order.

    With ``fuse``, q|k|v and gate|up (which share their input in a decoder) are quantized as one
    weight over concatenated output columns and run as one GEMV each (4 launches per layer);
    quantization is per column, so their codes, scales and zeros are those of the separate
    projections.

    With ``chain``, the whole pass is one ``laq_gemm_chain`` launch (M <= 4) whose stages follow
    the decoder's data flow: an entry waits for every earlier one unless it reads the input of
    the projection before it (k and v after q, up after gate), so each layer has the four
    dependency points q|k|v -> o -> gate|up -> down -> next layer.

    With ``planned`` (M <= 4), the same entries run through ``laq_pass_run`` after
    ``laq_pass_prepare`` has laid their weights out as per-SM streams (``_lib.PassPlan``)."""

    def __init__(self, model="qwen3-4b", bits=3, M=1, layers=inputs.LAYERS, seed=0,
                 outliers=False, device="cuda", pdl=True, fuse=False, chain=False,
                 planned=False):
        if planned and not 1 <= M <= 4:
            raise ValueError("the planned pass runs M = 1..4")
        self.model, self.bits, self.M, self.layers = model, bits, M, layers
        self.seed, self.outliers, self.fuse, self.chain = seed, outliers, fuse, chain
        self.planned = planned
        self.device = torch.device(device)
        plan = pass_plan(model, fuse, layers)
        xs = sum(M * K for *_, K, N in plan)
        ys = sum(M * N for *_, K, N in plan)
        self.Xbuf = torch.empty((xs,), dtype=torch.float16, device=self.device)
        self.Ybuf = torch.zeros((ys,), dtype=torch.float16, device=self.device)
        self.linears = []   # [(layer, member projection indices, name, QuantLinear)]
        self.X, self.Y = [], []
        xo = yo = 0
        for layer, members, name, K, N in plan:
            W = self.weight(layer, members)
            self.linears.append((layer, members, name, QuantLinear(W, bits)))
            del W
            x = self.Xbuf[xo:xo + M * K].view(M, K)
            x.copy_(inputs.activations_torch(M, K, inputs.proj_seed(seed, layer, members[0]),
                                             self.device))
            self.X.append(x)
            self.Y.append(self.Ybuf[yo:yo + M * N].view(M, N))
            xo += M * K
            yo += M * N
        # The library's own plan for each shape; with pdl, each launch may start (and prefetch
        # its weights, which no kernel of the pass writes) while the previous one finishes.
        sms = torch.cuda.get_device_properties(self.device).multi_processor_count
        self.configs = []
        for *_, q in self.linears:
            c = _lib.laq_gemm_plan(M, q.K, q.N, bits, sms)
            c.pdl = 1 if pdl else 0
            self.configs.append(c)
        if chain or planned:
            entries = []
            for i, (_, members, name, q) in enumerate(self.linears):
                wait = not (name in SHARES_INPUT and i > 0)
                entries.append((self.X[i], q.packed, q.s, q.z, bits, self.Y[i], wait))
            if planned:
                self.plan = _lib.PassPlan(entries, self.device)
                self.ws = self.plan.ws
            else:
                self.chain_spec = _lib.Chain(entries)
                self.ws = _lib.chain_workspace(len(entries), self.device)
        torch.cuda.synchronize(self.device)

    def weight(self, layer, members):
        """The fp16 weight of one launch (its member projections side by side), regenerated
        from their seeds."""
        if isinstance(members, int):
            members = (members,)
        parts = []
        for pi in members:
            _, K, N = shapes(self.model)[pi]
            parts.append(inputs.weights_torch(K, N, inputs.proj_seed(self.seed, layer, pi),
                                              self.device, outliers=self.outliers))
        return parts[0] if len(parts) == 1 else torch.cat(parts, dim=1)

    @property
    def launches(self):
        return 1 if self.chain or self.planned else len(self.linears)

    def bytes_per_pass(self):
        return sum(q.bytes_per_call(self.M) for *_, q in self.linears)

    def set_configs(self, configs):
        self.configs = list(configs)

    def run(self, stream=None, events=None):
        """Launch the pass; with ``events`` (launches + 1 CUDA events) record one before each
        launch and one after the last."""
        if self.chain or self.planned:
            if events is not None:
                events[0].record(stream)
            if self.planned:
                self.plan.run(stream)
            else:
                self.chain_spec.run(self.ws, stream)
            if events is not None:
                events[-1].record(stream)
            return
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
