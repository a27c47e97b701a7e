"""One form of the decode-step weight pass, replayed a few times: the case for profiling a pass.

    python -m paper_2605_08755_gb300.pass_case --variant graph_fused --layers 2 --replays 1

Builds the Qwen3-4B-shaped pass (synthetic weights; use a 1- or 2-layer pass under a profiler)
in one of its forms (``graph_252``, ``graph_fused``, ``chain_252``, ``chain_fused``, and the
planned pass over per-SM weight streams, ``planned_252`` and ``planned_fused``, M <= 4),
captures it into a CUDA graph (the capture is preceded by one eager run of the pass), replays
the graph ``replays`` times and prints the mean device time per replay.  Under a profiler, the
first replay's kernels follow the eager run's: for a graph form with L launches per pass,
``-k regex:gemm_kernel -s L -c 4`` selects one launch of each projection of the replay's first
layer; for a chain form ``-k regex:chain_kernel -s 1 -c 1`` and for a planned form
``-k regex:pass_kernel -s 1 -c 1`` select the replay's single launch.
""""""
import argparse
import json

import torch

from .weight_pass import WeightPass

VARIANTS = {"graph_252": (False, False, False), "graph_fused": (True, False, False),
            "chain_252": (False, True, False), "chain_fused": (True, True, False),
            "planned_252": (False, False, True), "planned_fused": (True, False, True)}


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--variant", default="graph_fused", choices=sorted(VARIANTS))
    ap.add_argument("--model", default="qwen3-4b", choices=["qwen3-4b", "qwen3-8b"])
    ap.add_argument("--bits", type=int, default=3, choices=[3, 4])
    ap.add_argument("--M", type=int, default=1)
    ap.add_argument("--layers", type=int, default=36)
    ap.add_argument("--replays", type=int, default=3)
    a = ap.parse_args()
    fuse, chain, planned = VARIANTS[a.variant]
    dev = torch.device("cuda", 0)
    torch.cuda.set_device(dev)
    wp = WeightPass(model=a.model, bits=a.bits, M=a.M, layers=a.layers, device=dev,
                    outliers=(a.model == "qwen3-8b"), fuse=fuse, chain=chain,
                    planned=planned)
    stream = torch.cuda.Stream(dev)
    g = wp.capture(stream=stream)
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    with torch.cuda.stream(stream):
        e0.record(stream)
        for _ in range(a.replays):
            g.replay()
        e1.record(stream)
    torch.cuda.synchronize(dev)
    us = e0.elapsed_time(e1) * 1e3 / a.replays
    print(json.dumps({"variant": a.variant, "bits": a.bits, "M": a.M, "layers": a.layers,
                      "launches": wp.launches, "bytes_per_pass": wp.bytes_per_pass(),
                      "us_per_pass": us, "gbs": wp.bytes_per_pass() / (us * 1e-6) / 1e9,
                      "configs": [c.as_dict() for c in wp.configs[:4 if fuse else 7]]}))


if __name__ == "__main__":
    main()
