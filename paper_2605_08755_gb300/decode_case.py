"""Time one whole decode step (DecodeStep) and, for context, the same step in fp16 torch ops.

    python -m paper_2605_08755_gb300.decode_case --bits 3 --M 1 --context 2048 [--fp16]
        [--rotation-rounds R]

Prints one JSON line: microseconds per step (CUDA events around graph replays on the capture
stream), tokens per second (M per step), the step's algorithmic bytes and GB/s, the weight pass
alone (the fused projections graph), and with --fp16 the same decoder step as a CUDA graph of
plain torch fp16 operations on the unquantized weights (F.rms_norm, matmul, rotary by hand,
scaled_dot_product_attention with grouped kv heads, SiLU, matmul with the embedding): a context
ratio like the paper's decode speed-up over FP16 (Sec. 5.2), measured here on one GB300.  With
--rotation-rounds R the line also times the rotation-based variant of the same step (an online
pairwise rotation of R rounds before every projection of a layer, norms unfused) and reports
how much faster the step is without it, the comparison of Sec. 5.2 (LAQuant against ParoQuant).
"""
import argparse
import json
import math

import torch

from .decode_step import DecodeStep


def time_graph(g, stream, replays):
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    with torch.cuda.stream(stream):
        for _ in range(3):
            g.replay()
        e0.record(stream)
        for _ in range(replays):
            g.replay()
        e1.record(stream)
    torch.cuda.synchronize()
    return e0.elapsed_time(e1) * 1e3 / replays


class Fp16Step:
    """The same decoder step in torch fp16 ops, weights unquantized (W regenerated from the
    seeds of ``st``), sharing st's embedding, norm weights and (copies of) its KV caches."""

    def __init__(self, st):
        import torch.nn.functional as F
        self.F, self.st = F, st
        self.W = [[st.wp.weight(l, members) for (_, members, _, _) in
                   st.wp.linears[4 * l:4 * l + 4]] for l in range(st.layers)]
        self.kc = [c.clone() for c in st.kc]
        self.vc = [c.clone() for c in st.vc]
        D, p = st.D, st.context - 1
        i = torch.arange(D // 2, device=st.device, dtype=torch.float32)
        a = p * st.theta ** (-2.0 * i / D)
        self.cos = torch.cat([a.cos(), a.cos()]).to(torch.float16)
        self.sin = torch.cat([-a.sin(), a.sin()]).to(torch.float16)

    def rope(self, x):
        D = x.shape[-1]
        rot = torch.cat([x[..., D // 2:], x[..., :D // 2]], dim=-1)
        return x * self.cos + rot * self.sin

    def run(self):
        st, F = self.st, self.F
        M, H, Hq, Hkv, D, I, eps = st.M, st.H, st.Hq, st.Hkv, st.D, st.I, st.eps
        p = st.context - 1
        x = st.E[st.tokens.long()]
        r = x
        h = F.rms_norm(x, (H,), st.norms[0]["in_w"], eps)
        d = None
        for l in range(st.layers):
            nw, (Wqkv, Wo, Wgu, Wd) = st.norms[l], self.W[l]
            if l > 0:
                r = r + d
                h = F.rms_norm(r, (H,), nw["in_w"], eps)
            qkv = h @ Wqkv
            q = qkv[:, :Hq * D].view(M, Hq, D)
            k = qkv[:, Hq * D:(Hq + Hkv) * D].view(M, Hkv, D)
            v = qkv[:, (Hq + Hkv) * D:].view(M, Hkv, D)
            q = self.rope(F.rms_norm(q, (D,), nw["q_w"], eps))
            k = self.rope(F.rms_norm(k, (D,), nw["k_w"], eps))
            self.kc[l][:, :, p] = k
            self.vc[l][:, :, p] = v
            a = F.scaled_dot_product_attention(q.view(M, Hq, 1, D), self.kc[l], self.vc[l],
                                               enable_gqa=True)
            o = a.reshape(M, Hq * D) @ Wo
            r = r + o
            h = F.rms_norm(r, (H,), nw["post_w"], eps)
            gu = h @ Wgu
            d = (F.silu(gu[:, :I]) * gu[:, I:]) @ Wd
        r = r + d
        h = F.rms_norm(r, (H,), st.final_w, eps)
        return torch.argmax(h @ st.E.t(), dim=1)

    def capture(self, stream):
        self.run()
        torch.cuda.synchronize()
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g, stream=stream):
            self.run()
        return g


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--model", default="qwen3-4b", choices=["qwen3-4b", "qwen3-8b"])
    ap.add_argument("--bits", type=int, default=3, choices=[3, 4])
    ap.add_argument("--M", type=int, default=1)
    ap.add_argument("--layers", type=int, default=36)
    ap.add_argument("--context", type=int, default=2048)
    ap.add_argument("--replays", type=int, default=50)
    ap.add_argument("--fp16", action="store_true")
    ap.add_argument("--separate-attention", action="store_true")
    ap.add_argument("--separate-norms", action="store_true")
    ap.add_argument("--rotation-rounds", type=int, default=0)
    a = ap.parse_args()
    torch.cuda.set_device(0)
    st = DecodeStep(model=a.model, bits=a.bits, M=a.M, layers=a.layers, context=a.context,
                    fused_attention=not a.separate_attention, fused_norms=not a.separate_norms)
    stream = torch.cuda.Stream()
    g = st.capture(stream=stream)
    us = time_graph(g, stream, a.replays)
    gw = st.wp.capture(stream=stream)
    us_w = time_graph(gw, stream, a.replays)
    del gw
    out = {"model": a.model, "bits": a.bits, "M": a.M, "layers": a.layers,
           "context": a.context, "launches": st.launches, "us_per_step": us,
           "tokens_per_s": a.M / (us * 1e-6), "bytes_per_step": st.bytes_per_step(),
           "gbs": st.bytes_per_step() / (us * 1e-6) / 1e9, "weight_pass_us": us_w}
    del g
    if a.rotation_rounds:
        rs = DecodeStep(model=a.model, bits=a.bits, M=a.M, layers=a.layers, context=a.context,
                        fused_attention=not a.separate_attention,
                        rotation_rounds=a.rotation_rounds)
        gr = rs.capture(stream=stream)
        us_rot = time_graph(gr, stream, a.replays)
        out.update({"rotation_rounds": a.rotation_rounds, "rotated_launches": rs.launches,
                    "rotated_us_per_step": us_rot,
                    "speedup_without_rotation": us_rot / us - 1.0})
        del gr, rs
    if a.fp16:
        ref = Fp16Step(st)
        gr = ref.capture(stream)
        us16 = time_graph(gr, stream, a.replays)
        out.update({"fp16_torch_us_per_step": us16, "speedup_vs_fp16": us16 / us})
    print(json.dumps(out), flush=True)


if __name__ == "__main__":
    main()
