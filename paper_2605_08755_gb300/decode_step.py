"""One decode step of a Qwen3-shaped decoder with WbG128 projections, on the library's kernels.

The decode step whose speed Sec. 5.2 reports, with synthetic weights: the embedding gather, then
per layer

    h = rmsnorm(r)                      (r: the residual stream; layer 0: r = x)
    q, k, v = q|k|v GEMV(h); q, k = rope(rmsnorm(q)), rope(rmsnorm(k)); k, v -> cache at pos
    a = attention(q, cache[: pos + 1])  (grouped-query)
    h = rmsnorm(r += o GEMV(a))
    d = down GEMV(silu(gate) * up),  gate|up = gate|up GEMV(h);  r += d  (in the next norm)

then the final rmsnorm, the LM head (the embedding, tied as in Qwen3-4B, quantized like the
projections) and the greedy argmax.  With ``rotation_rounds`` > 0 the step is that of a
rotation-based quantizer instead: the input of every projection of a layer first goes through
the online pairwise rotation (``laq_pairwise_rotate``: channel scales and that many rounds of
Givens rotations per 128-channel group, synthetic tables), the per-token work LAQuant removes
(Sec. 5.2 measures decoding with and without it).  Every step of it runs in the library's kernels
(``laq_gemm_wxg128`` and the decoder operations of include/laq.h), launched in stream order
with programmatic dependent launch and captured into one CUDA graph.  The KV cache holds
``context - 1`` synthetic tokens before the new one, so attention reads ``context`` tokens.
"""
import math

import torch

from . import _lib, inputs
from .weight_pass import QuantLinear, WeightPass


class DecodeStep:
    def __init__(self, model="qwen3-4b", bits=3, M=1, layers=inputs.LAYERS, context=2048,
                 vocab=None, seed=0, device="cuda", fused_attention=True, fused_norms=True,
                 rotation_rounds=0):
        dims = inputs.DECODER[model]
        self.model, self.bits, self.M, self.layers = model, bits, M, layers
        self.fused_attention = fused_attention
        # the layers' RMSNorms folded into the next GEMV (not with a rotation between them)
        self.fused_norms = fused_norms and not rotation_rounds
        self.rotation_rounds = rotation_rounds
        self.context, self.seed = context, seed
        self.H, self.Hq, self.Hkv, self.D, self.I = (dims[k] for k in ("H", "Hq", "Hkv", "D", "I"))
        self.V = vocab or dims["V"]
        self.theta, self.eps = dims["theta"], dims["eps"]
        self.device = dev = torch.device(device)
        H, Hq, Hkv, D, I, V = self.H, self.Hq, self.Hkv, self.D, self.I, self.V

        # projections: the fused q|k|v, o, gate|up, down of each layer, with their launch plans
        self.wp = WeightPass(model=model, bits=bits, M=M, layers=layers, seed=seed, device=dev,
                             outliers=(model == "qwen3-8b"), fuse=True)
        self.proj = [[q for *_, q in self.wp.linears[4 * l:4 * l + 4]] for l in range(layers)]
        self.cfg = [self.wp.configs[4 * l:4 * l + 4] for l in range(layers)]
        self.norms = []
        for l in range(layers):
            base = inputs.proj_seed(seed, l, 10)
            self.norms.append({"in_w": inputs.norm_weight_torch(H, base, dev),
                               "post_w": inputs.norm_weight_torch(H, base + 1, dev),
                               "q_w": inputs.norm_weight_torch(D, base + 2, dev),
                               "k_w": inputs.norm_weight_torch(D, base + 3, dev)})
        self.final_w = inputs.norm_weight_torch(H, inputs.proj_seed(seed, layers, 10), dev)
        self.E = inputs.embedding_torch(V, H, seed, dev)
        self.lm = QuantLinear(self.E.t().contiguous(), bits)     # [H, V]
        self.lm_cfg = _lib.laq_gemm_plan(M, H, V, bits,
                                         torch.cuda.get_device_properties(dev).multi_processor_count)
        self.lm_cfg.pdl = 1

        # the KV cache: context - 1 synthetic tokens, the new one goes to position context - 1
        self.kc = [inputs.kv_cache_torch(M, Hkv, context, D, inputs.proj_seed(seed, l, 20), dev)
                   for l in range(layers)]
        self.vc = [inputs.kv_cache_torch(M, Hkv, context, D, inputs.proj_seed(seed, l, 21), dev)
                   for l in range(layers)]
        self.tokens = torch.from_numpy(inputs.tokens(M, V, seed)).to(dev)
        self.pos = torch.full((M,), context - 1, dtype=torch.int32, device=dev)
        self.lens = self.pos + 1

        f16 = dict(dtype=torch.float16, device=dev)
        self.x = torch.empty((M, H), **f16)
        self.r = torch.empty((M, H), **f16)
        self.r2 = torch.empty((M, H), **f16)  # the residual's other buffer (fused norms)
        self.h = torch.empty((M, H), **f16)
        self.qkv = torch.empty((M, (Hq + 2 * Hkv) * D), **f16)
        self.q = torch.empty((M, Hq, D), **f16)
        self.att = torch.empty((M, Hq, D), **f16)
        self.o = torch.empty((M, H), **f16)
        self.gu = torch.empty((M, 2 * I), **f16)
        self.act = torch.empty((M, I), **f16)
        self.d = torch.empty((M, H), **f16)
        self.logits = torch.empty((M, V), **f16)
        self.next = torch.empty((M,), dtype=torch.int32, device=dev)
        self.ws = (_lib.attention_qkv_workspace(M, Hq, Hkv, context, dev) if fused_attention
                   else _lib.attention_workspace(M, Hq, context, dev))
        self.scale = 1.0 / math.sqrt(D)

        # the rotation-based variant: per layer, tables for the inputs of q|k|v, o, gate|up, down
        self.rot = []
        if rotation_rounds:
            for l in range(layers):
                tabs = {}
                for j, (name, K) in enumerate((("qkv", H), ("o", Hq * D), ("gate_up", H),
                                               ("down", I))):
                    pairs, theta, alpha = inputs.rotation(K, rotation_rounds,
                                                          inputs.proj_seed(seed, l, 30 + j))
                    th = torch.from_numpy(theta).to(dev)
                    tabs[name] = dict(pairs=torch.from_numpy(pairs).to(dev), theta=th,
                                      cs=_lib.laq_rotation_tables(th),
                                      alpha=torch.from_numpy(alpha).to(dev))
                self.rot.append(tabs)
            self.xr = {K: torch.empty((M, K), **f16) for K in {H, Hq * D, I}}

    def gemv(self, X, q, Y, cfg, stream, rot=None):
        X = X.view(self.M, -1)
        if rot is not None:  # the rotation-based variant: turn the input first
            Xr = self.xr[X.shape[1]]
            _lib.laq_pairwise_rotate(X, rot["pairs"], rot["cs"], alpha=rot["alpha"], Y=Xr,
                                     stream=stream)
            X = Xr
        _lib.laq_gemm_wxg128(X, q.packed, q.s, q.z, q.bits, Y=Y.view(self.M, -1), config=cfg,
                             stream=stream)

    def run(self, stream=None):
        """Launch one step on ``stream``: reads tokens, pos, the caches; writes the caches at pos,
        logits and next (the greedy tokens)."""
        if self.fused_norms:
            return self.run_fused(stream)
        L = _lib
        _lib.laq_embed(self.E, self.tokens, X=self.x, stream=stream)
        L.laq_rmsnorm(self.x, self.norms[0]["in_w"], self.eps, R_out=self.r, Y=self.h,
                      stream=stream)
        for l in range(self.layers):
            nw, (qkv, o, gu, dn), cf = self.norms[l], self.proj[l], self.cfg[l]
            rt = self.rot[l] if self.rot else {}
            if l > 0:
                L.laq_rmsnorm(self.d, nw["in_w"], self.eps, R=self.r, R_out=self.r, Y=self.h,
                              stream=stream)
            self.gemv(self.h, qkv, self.qkv, cf[0], stream, rt.get("qkv"))
            if self.fused_attention:  # norm, rotation, cache append and attention: two launches
                L.laq_attention_qkv(self.qkv, nw["q_w"], nw["k_w"], self.pos, self.Hq, self.Hkv,
                                    self.theta, self.eps, self.kc[l], self.vc[l], self.scale,
                                    self.ws, out=self.att, stream=stream)
            else:
                L.laq_qk_norm_rope(self.qkv, nw["q_w"], nw["k_w"], self.pos, self.Hq, self.Hkv,
                                   self.theta, self.eps, self.kc[l], self.vc[l], q_out=self.q,
                                   stream=stream)
                L.laq_attention_decode(self.q, self.kc[l], self.vc[l], self.lens, self.scale,
                                       self.ws, out=self.att, stream=stream)
            self.gemv(self.att, o, self.o, cf[1], stream, rt.get("o"))
            L.laq_rmsnorm(self.o, nw["post_w"], self.eps, R=self.r, R_out=self.r, Y=self.h,
                          stream=stream)
            self.gemv(self.h, gu, self.gu, cf[2], stream, rt.get("gate_up"))
            L.laq_silu_mul(self.gu, h=self.act, stream=stream)
            self.gemv(self.act, dn, self.d, cf[3], stream, rt.get("down"))
        L.laq_rmsnorm(self.d, self.final_w, self.eps, R=self.r, Y=self.h, stream=stream)
        self.gemv(self.h, self.lm, self.logits, self.lm_cfg, stream)
        L.laq_argmax(self.logits, out=self.next, stream=stream)

    def run_fused(self, stream=None):
        """The same step with the two RMSNorms of each layer (and their residual adds) folded into
        the X staging of the q|k|v and gate|up GEMVs (laq_gemm_wxg128_prologue); the residual
        alternates between two buffers, since a prologue's residual output may not alias its
        inputs.  SiLU*up and the final norm stay separate kernels: on GB300 their prologue forms
        measured slower (every CTA of the down GEMV recomputes SiLU over its K range before its
        first MMA; the LM head's ~1200 CTAs each redo the row norm)."""
        L = _lib
        RMS = _lib.PROLOGUE_RMSNORM
        L.laq_embed(self.E, self.tokens, X=self.x, stream=stream)
        res, nxt = self.r, self.r2
        for l in range(self.layers):
            nw, (qkv, o, gu, dn), cf = self.norms[l], self.proj[l], self.cfg[l]
            if l == 0:  # r = x
                L.laq_gemm_wxg128_prologue(self.x, qkv.packed, qkv.s, qkv.z, qkv.bits, RMS,
                                           Y=self.qkv, R_out=res, w=nw["in_w"], eps=self.eps,
                                           config=cf[0], stream=stream)
            else:       # r += d
                L.laq_gemm_wxg128_prologue(self.d, qkv.packed, qkv.s, qkv.z, qkv.bits, RMS,
                                           Y=self.qkv, R=res, R_out=nxt, w=nw["in_w"],
                                           eps=self.eps, config=cf[0], stream=stream)
                res, nxt = nxt, res
            L.laq_attention_qkv(self.qkv, nw["q_w"], nw["k_w"], self.pos, self.Hq, self.Hkv,
                                self.theta, self.eps, self.kc[l], self.vc[l], self.scale, self.ws,
                                out=self.att, stream=stream)
            self.gemv(self.att, o, self.o, cf[1], stream)
            L.laq_gemm_wxg128_prologue(self.o, gu.packed, gu.s, gu.z, gu.bits, RMS, Y=self.gu,
                                       R=res, R_out=nxt, w=nw["post_w"], eps=self.eps,
                                       config=cf[2], stream=stream)
            res, nxt = nxt, res
            L.laq_silu_mul(self.gu, h=self.act, stream=stream)
            self.gemv(self.act, dn, self.d, cf[3], stream)
        L.laq_rmsnorm(self.d, self.final_w, self.eps, R=res, Y=self.h, stream=stream)
        self.gemv(self.h, self.lm, self.logits, self.lm_cfg, stream)
        L.laq_argmax(self.logits, out=self.next, stream=stream)

    @property
    def launches(self):
        # embed, norm, per layer 4 GEMVs + 2 norms (1 in layer 0) + attention (2 fused, else
        # rope + 2) + silu, final norm, LM head, argmax
        if self.fused_norms:  # embed, per layer 4 GEMVs + 2 attention + silu, norm, LM head, argmax
            return 1 + self.layers * 7 + 3
        per_layer = (9 if self.fused_attention else 10) + (4 if self.rotation_rounds else 0)
        return 2 + self.layers * per_layer - 1 + 3

    def capture(self, stream=None):
        self.run()
        torch.cuda.synchronize(self.device)
        g = torch.cuda.CUDAGraph()
        s = torch.cuda.Stream(self.device) if stream is None else stream
        with torch.cuda.graph(g, stream=s):
            self.run(stream=s)
        return g

    def bytes_per_step(self):
        """Algorithmic HBM bytes of one step: the projections and the LM head (packed codes, s,
        z, X, Y), the KV cache read (context tokens of k and v per layer) and written (the new
        token), and the embedding row."""
        M, D, Hkv = self.M, self.D, self.Hkv
        kv = self.layers * M * Hkv * D * 2 * 2 * (self.context + 1)
        return (self.wp.bytes_per_pass() + self.lm.bytes_per_call(M) + kv + M * self.H * 2)
