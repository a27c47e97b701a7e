"""One projection's GEMV, launched a few times: the small case for profiling a single kernel.

    python -m paper_2605_08755_gb300.gemv_case --K 2560 --N 9728 --bits 3 --M 1 --iters 5

Quantizes and packs one synthetic weight (seeded, as in the decode-step pass), launches
``laq_gemm_wxg128`` twice to warm up, then ``iters`` times back to back on one stream with the
library's own launch plan, and prints the plan and the mean CUDA-event time per timed launch
(the weight, 10 MB for the default gate shape, stays in L2 between launches, so this is a
warm-L2 figure).  Under a profiler, ``-k regex:gemm_kernel -s 2 -c 1`` picks the first timed
launch (the skip count applies to the launches the name filter matches).
"""
import argparse
import json

import torch

from . import _lib, inputs


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--K", type=int, default=2560)
    ap.add_argument("--N", type=int, default=9728)
    ap.add_argument("--bits", type=int, default=3, choices=[3, 4])
    ap.add_argument("--M", type=int, default=1)
    ap.add_argument("--iters", type=int, default=5)
    ap.add_argument("--seed", type=int, default=4)
    a = ap.parse_args()
    dev = torch.device("cuda", 0)
    torch.cuda.set_device(dev)
    W = inputs.weights_torch(a.K, a.N, a.seed, dev)
    X = inputs.activations_torch(a.M, a.K, a.seed, dev)
    codes, s, z = _lib.laq_quantize_rtn(W, a.bits)
    packed = _lib.laq_pack(codes, a.bits)
    del W, codes
    Y = torch.empty((a.M, a.N), dtype=torch.float16, device=dev)
    cfg = _lib.laq_gemm_plan(a.M, a.K, a.N, a.bits,
                             torch.cuda.get_device_properties(dev).multi_processor_count)
    stream = torch.cuda.current_stream(dev)
    for _ in range(2):
        _lib.laq_gemm_wxg128(X, packed, s, z, a.bits, Y=Y, config=cfg, stream=stream)
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    for _ in range(a.iters):
        _lib.laq_gemm_wxg128(X, packed, s, z, a.bits, Y=Y, config=cfg, stream=stream)
    e1.record(stream)
    torch.cuda.synchronize(dev)
    nbytes = (a.K * a.N * a.bits // 8 + (a.K // 128) * a.N * 3 + 2 * a.M * a.K
              + 2 * a.M * a.N)
    us = e0.elapsed_time(e1) * 1e3 / a.iters
    print(json.dumps({"K": a.K, "N": a.N, "bits": a.bits, "M": a.M, "config": cfg.as_dict(),
                      "bytes_per_launch": nbytes, "us_per_launch": us,
                      "gbs": nbytes / (us * 1e-6) / 1e9}))


if __name__ == "__main__":
    main()
