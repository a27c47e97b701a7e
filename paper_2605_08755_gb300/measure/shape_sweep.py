"""Launch shapes of laq_gemm_wxg128 inside a whole decode-step weight pass, per projection.

For one fused 36-layer pass (q|k|v, o, gate|up, down; Qwen3-4B or Qwen3-8B shapes, W3 or W4,
batch rows M) captured as one CUDA graph, every launch shape (tiles per CTA, warps, cluster)
of one projection type is tried in turn -- the other projections keep the library's plan, the
ring depth follows the library's rule for the shape -- and the pass is timed (CUDA events on
the replaying stream, best of three runs of 100 replays).  Prints the library's shape and the
fastest shapes for each projection type, then the pass with every type at its fastest.

    python -m paper_2605_08755_gb300.measure.shape_sweep --model qwen3-8b --bits 3 --M 1
"""
import argparse
import itertools
import json
import os
import sys


def ring_stages(K, nt, warps, cl, bits):
    """(warps launched, ring stages) the library's rule gives a shape."""
    G = K // 128
    rec = 1024 if bits == 4 else 768
    gc = -(-G // cl)
    wt = max(1, min(gc, warps // nt))
    w = wt * nt
    st = min(16, max(2, -(-gc // wt) + 1))
    while st > 2 and w * st * rec > 100 * 1024:
        st -= 1
    return w, st


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--model", default="qwen3-4b", choices=["qwen3-4b", "qwen3-8b"])
    ap.add_argument("--bits", type=int, default=3, choices=[3, 4])
    ap.add_argument("--M", type=int, default=1)
    ap.add_argument("--json", default=None, help="write every timing to this file")
    a = ap.parse_args()
    root = os.path.abspath(os.path.join(os.path.dirname(__file__), "..", ".."))
    sys.path.insert(0, root)
    import torch

    import bench
    from paper_2605_08755_gb300 import _lib
    from paper_2605_08755_gb300.weight_pass import WeightPass

    dev = torch.device("cuda", 0)
    stream = torch.cuda.Stream()
    sms = torch.cuda.get_device_properties(dev).multi_processor_count
    wp = WeightPass(model=a.model, bits=a.bits, M=a.M, device=dev, fuse=True,
                    outliers=a.model == "qwen3-8b")
    base = list(wp.configs)
    names = [name for _, _, name, _ in wp.linears]

    def timed(cfgs):
        wp.set_configs(cfgs)
        g = wp.capture(stream=stream)
        t = min(bench.time_graph(g, stream, 100, dev) for _ in range(3)) * 1e3
        del g
        return t

    def config(q, nt, w, cl, st):
        c = _lib.laq_gemm_plan(a.M, q.K, q.N, a.bits, sms)
        c.tiles_per_cta, c.warps, c.cluster, c.stages, c.pdl = nt, w, cl, st, 1
        return c

    out = {"model": a.model, "bits": a.bits, "M": a.M, "library_us": timed(base), "types": {}}
    print(f"{a.model} W{a.bits} M={a.M}: library plan {out['library_us']:.1f} us per pass",
          flush=True)
    best = {}
    for ty in ("qkv", "o", "gate_up", "down"):
        idx = [i for i, n in enumerate(names) if n == ty]
        q = wp.linears[idx[0]][3]
        res = []
        for nt, warps, cl in itertools.product((1, 2, 4, 8), (4, 8, 16) if a.M >= 3 else (4, 8),
                                               (1, 2, 4, 8)):
            if warps % nt or cl > q.K // 128 or -(-(q.N // 16) // nt) * cl > 16 * sms:
                continue
            w, st = ring_stages(q.K, nt, warps, cl, a.bits)
            cfgs = list(base)
            for i in idx:
                cfgs[i] = config(q, nt, w, cl, st)
            try:
                res.append((timed(cfgs), nt, w, cl, st))
            except _lib.LaqError:
                continue   # more shared memory than a CTA may have
        res.sort()
        b = base[idx[0]]
        lib = (b.tiles_per_cta, b.warps, b.cluster, b.stages)
        out["types"][ty] = {"K": q.K, "N": q.N, "library": lib, "timings": res}
        print(f"  {ty:8s} K={q.K:5d} N={q.N:5d} library {lib}  fastest "
              + ", ".join(f"{r[0]:.1f} {tuple(r[1:4])}" for r in res[:4]),
              flush=True)
        best[ty] = (q, res[0])
    cfgs = list(base)
    for ty, (q, (t, nt, w, cl, st)) in best.items():
        for i, n in enumerate(names):
            if n == ty:
                cfgs[i] = config(q, nt, w, cl, st)
    out["fastest_us"] = timed(cfgs)
    print(f"  every type at its fastest shape: {out['fastest_us']:.1f} us "
          f"(library {timed(base):.1f})", flush=True)
    if a.json:
        with open(a.json, "w") as f:
            json.dump(out, f)


if __name__ == "__main__":
    main()
