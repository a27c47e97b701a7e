"""Benchmark: the Qwen3-shaped decode-step weight pass (W3G128 by default) on GB300.

One step = one replay of a CUDA graph holding every quantized projection of the model once
(36 layers x q, k, v, o, gate, up, down, M = 1), i.e. the weight streaming of one batch-1
decode step.  The pass has four equivalent forms (252 ``laq_gemm_wxg128`` launches; 144 with
q|k|v and gate|up fused over concatenated columns; one persistent ``laq_gemm_chain`` launch of
either list); each is timed briefly and the fastest gets the full timed run.  Quantization and packing (``laq_quantize_rtn``,
``laq_pack``) are the offline model-preparation steps and run once before timing; their time is
reported as ``prep_ms``.  Synthetic weights ~ N(0, 0.02^2) and activations ~ N(0, 1) stand in
for the paper's Qwen3 checkpoints.

Prints one JSON line.  ``value`` is the achieved HBM bandwidth of the pass (algorithmic bytes =
packed codes + s + z + X + Y, per step, all ranks) over the device time of the timed replays.

    python bench.py [--steps K] [--warmup W] [--model qwen3-4b|qwen3-8b] [--bits 3|4] [--M 1]
    python bench.py --impl reference      # the CPU oracle, timed on the host cores
    torchrun --nproc-per-node N bench.py --gpus N   # N independent replicas (no data exchange)
"""
import argparse
import json
import os
import statistics
import subprocess
import sys
import tempfile
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

METRIC = "W3G128 dequant-GEMV HBM GB/s (% of peak); µs per Qwen3-4B-shaped decode step"


def parse():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=4000)
    ap.add_argument("--warmup", type=int, default=20)
    ap.add_argument("--impl", default="laq", choices=["laq", "reference"])
    ap.add_argument("--model", default="qwen3-4b", choices=["qwen3-4b", "qwen3-8b"])
    ap.add_argument("--bits", type=int, default=3, choices=[3, 4])
    ap.add_argument("--M", type=int, default=1)
    ap.add_argument("--layers", type=int, default=36)
    ap.add_argument("--no-fp16", action="store_true", help="skip the fp16 torch.matmul context")
    ap.add_argument("--cpu-seconds", type=float, default=12.0,
                    help="CPU work budget of the oracle baseline sample")
    return ap.parse_args()


def workload_name(a):
    return (f"{a.model} decode-step weight pass, {a.layers} layers x 7 projections, "
            f"W{a.bits}G128, M={a.M}, one CUDA graph")


def load_peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        with open(p) as f:
            d = json.load(f)
        return float(d["hbm_gbs"]), "measured"
    return 6800.0, "fallback"


def traffic_for(kernel, a, variant, shapes=None):
    """DRAM bytes per launch of ``kernel`` in pass form ``variant``, measured by ncu
    (profiles/traffic.json), or None when no capture exists for this kernel and workload, the
    kernel's source changed since, or the instance now runs other projections (``shapes``: the
    sorted [K, N, launches] of its launches in one step)."""
    import hashlib
    path = os.path.join(ROOT, "profiles", "traffic.json")
    if not os.path.exists(path):
        return None
    with open(path) as f:
        table = json.load(f)
    entry = table.get(f"{kernel} {a.model} W{a.bits} M={a.M} {variant}")
    if not entry:
        return None
    if shapes is not None and entry.get("shapes") != shapes:
        return None
    h = hashlib.sha256()
    for name in entry["sources"]:
        with open(os.path.join(ROOT, "paper_2605_08755_gb300", "csrc", name), "rb") as f:
            h.update(f.read())
    return entry["dram_bytes_per_launch"] if h.hexdigest() == entry["sources_sha256"] else None


# ------------------------------------------------------------------ distributed plumbing


def dist_setup(a):
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    if world > 1:
        import torch.distributed as dist
        backend = "nccl" if a.impl == "laq" else "gloo"
        if backend == "nccl":
            import torch
            torch.cuda.set_device(local)
        dist.init_process_group(backend=backend)
    return world, rank, local


def barrier(world):
    if world > 1:
        import torch.distributed as dist
        dist.barrier()


def max_over_ranks(world, value, device=None):
    if world == 1:
        return value
    import torch
    import torch.distributed as dist
    t = torch.tensor([value], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def sum_over_ranks(world, value, device=None):
    if world == 1:
        return value
    import torch
    import torch.distributed as dist
    t = torch.tensor([value], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.SUM)
    return float(t.item())


# ------------------------------------------------------------------ clocks


class ClockSampler:
    """nvidia-smi samples of SM clock and throttle reasons while the timed region runs."""

    Q = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
         "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
         "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index):
        self.gpu = gpu_index
        self.proc = None
        self.out = None

    def __enter__(self):
        try:
            self.out = tempfile.NamedTemporaryFile("w+", suffix=".csv", delete=False)
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--query-gpu={self.Q}", "--format=csv,noheader,nounits",
                 "-i", str(self.gpu), "-lms", "100"], stdout=self.out,
                stderr=subprocess.DEVNULL)
        except (OSError, ValueError):
            self.proc = None
        time.sleep(0.3)
        return self

    def __exit__(self, *exc):
        if self.proc is not None:
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except subprocess.TimeoutExpired:
                self.proc.kill()

    def summary(self):
        if self.proc is None or self.out is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        self.out.flush()
        rows = []
        with open(self.out.name) as f:
            for line in f:
                parts = [p.strip() for p in line.split(",")]
                if len(parts) < 9:
                    continue
                try:
                    rows.append((float(parts[1]), float(parts[2]), float(parts[3]), parts[4:]))
                except ValueError:
                    continue
        os.unlink(self.out.name)
        if not rows:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["no samples"]}
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = set()
        for *_, flags in rows:
            for n, v in zip(names, flags[1:]):
                if v.strip().lower() == "active":
                    reasons.add(n)
        loaded = [r for r in rows if r[2] > 0] or rows
        return {"sm_mhz": statistics.median(r[0] for r in loaded),
                "sm_max_mhz": max(r[1] for r in rows), "reasons": sorted(reasons),
                "samples": len(rows), "power_w_max": max(r[2] for r in rows)}


# ------------------------------------------------------------------ CPU oracle baseline


class OracleSample:
    """A bounded sample of the same workload for the C oracle: the projections of layer 0 (same
    shapes, distributions and seeds recipe), quantized once by the oracle (untimed).  ``run``
    times the oracle's fp64 dequantize-and-multiply over whole projections (or a leading
    column slice of one, when a short step is asked for)."""

    def __init__(self, model, bits, M, seed=0):
        from oracle import c_oracle
        from paper_2605_08755_gb300 import inputs
        from paper_2605_08755_gb300.weight_pass import shapes
        self.co = c_oracle
        self.bits, self.M = bits, M
        self.items = []
        for pi, (name, K, N) in enumerate(shapes(model)):
            sd = inputs.proj_seed(seed, 0, pi)
            W = inputs.weights(K, N, sd, outliers=(model == "qwen3-8b"))
            codes, s, z = c_oracle.quantize_rtn(W, bits)
            self.items.append((f"L0.{name}", codes, s, z, inputs.activations(M, K, sd)))
        self.next = 0

    def nbytes(self, K, N):
        return K * N * self.bits // 8 + (K // 128) * N * 3 + 2 * self.M * K + 2 * self.M * N

    def run(self, seconds, max_cols=None):
        """Oracle work for about ``seconds``; returns (bytes, seconds spent, items done)."""
        done = 0
        spent = 0.0
        names = []
        while True:   # at least one item
            name, codes, s, z, X = self.items[self.next % len(self.items)]
            self.next += 1
            K, N = codes.shape
            if max_cols is not None and max_cols < N:
                codes, s, z = (codes[:, :max_cols].copy(), s[:, :max_cols].copy(),
                               z[:, :max_cols].copy())
                N = max_cols
                name += f"[:, :{N}]"
            t0 = time.perf_counter()
            self.co.gemm(X, codes, s, z)
            spent += time.perf_counter() - t0
            done += self.nbytes(K, N)
            names.append(name)
            if spent >= seconds:
                break
        return done, spent, names


# ------------------------------------------------------------------ reference arm


def run_reference(a, world, rank):
    """The oracle, as it stands, on the host cores: each step is a bounded sample of the pass
    (a column slice of one projection, sized so the whole run stays within a few minutes)."""
    if rank != 0:
        return
    smp = OracleSample(a.model, a.bits, a.M)
    per_step_s = min(0.25, max(0.002, 90.0 / max(1, a.steps + a.warmup)))
    # calibrate columns per step on the first projection
    name, codes, *_ = smp.items[0]
    K, N = codes.shape
    b, sp, _ = smp.run(0.0, max_cols=64)
    cols = int(max(16, min(N, 64 * per_step_s / max(sp, 1e-6))) // 16 * 16)
    smp.next = 0
    for _ in range(a.warmup):
        smp.run(0.0, max_cols=cols)
    tot_b, tot_s, names = 0, 0.0, []
    step_s = []
    for _ in range(a.steps):
        b, sp, nm = smp.run(0.0, max_cols=cols)
        tot_b += b
        tot_s += sp
        step_s.append(sp)
        names += nm
    value = tot_b / tot_s / 1e9
    sample = (f"C oracle (fp64, one thread) dequantize-and-multiply; each step = the first "
              f"{cols} columns of one layer-0 projection, round-robin over q,k,v,o,gate,up,down; "
              f"{tot_s:.1f} s of CPU work over {a.steps} steps; quantization not timed")
    line = {"metric": METRIC, "value": value, "unit": "GB/s", "n_gpus": a.gpus,
            "steps": a.steps, "warmup": a.warmup,
            "ms_per_step": 1e3 * statistics.median(step_s), "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
            "impl": "reference", "config": {"workload": workload_name(a), "model": a.model},
            "cpu_baseline": {"value": value, "unit": "GB/s", "cores": 1, "kind": "oracle",
                             "sample": sample},
            "e2e": {"value": value, "unit": "GB/s", "h2d_bytes_per_step": 0,
                    "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)


# ------------------------------------------------------------------ GPU arm


def fp16_context(a, dev, steps=50):
    """Time torch.matmul in fp16 over the same 252 shapes in one CUDA graph (context ratio)."""
    import torch

    from paper_2605_08755_gb300 import inputs
    from paper_2605_08755_gb300.weight_pass import shapes
    Ws, Xs, Ys = [], [], []
    for layer in range(a.layers):
        for pi, (_, K, N) in enumerate(shapes(a.model)):
            sd = inputs.proj_seed(0, layer, pi)
            Ws.append(inputs.weights_torch(K, N, sd, dev))
            Xs.append(inputs.activations_torch(a.M, K, sd, dev))
            Ys.append(torch.empty((a.M, N), dtype=torch.float16, device=dev))

    def run():
        for W, X, Y in zip(Ws, Xs, Ys):
            torch.matmul(X, W, out=Y)

    run()
    torch.cuda.synchronize(dev)
    g = torch.cuda.CUDAGraph()
    s = torch.cuda.Stream(dev)
    with torch.cuda.graph(g, stream=s):
        run()
    for _ in range(5):
        g.replay()
    torch.cuda.synchronize(dev)
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record()
    for _ in range(steps):
        g.replay()
    e1.record()
    torch.cuda.synchronize(dev)
    us = e0.elapsed_time(e1) * 1e3 / steps
    nbytes = sum(W.numel() * 2 for W in Ws) + sum(X.numel() * 2 for X in Xs) + \
        sum(Y.numel() * 2 for Y in Ys)
    del Ws, Xs, Ys, g
    torch.cuda.empty_cache()
    return us, nbytes


def time_graph(graph, stream, reps, dev):
    """Device time (ms) of ``reps`` back-to-back replays, CUDA events on ``stream``."""
    import torch
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    with torch.cuda.stream(stream):
        graph.replay()
        e0.record(stream)
        for _ in range(reps):
            graph.replay()
        e1.record(stream)
    torch.cuda.synchronize(dev)
    return e0.elapsed_time(e1) / reps


def kernel_breakdown(wp, stream, dev, reps=200):
    """Per GEMM kernel instance (bits, M class, tiles per CTA): a CUDA graph of all of its
    launches of one step, in pass order, timed on the stream they run on; returns rows of
    (instance, launches, algorithmic bytes per step, us per step, [[K, N, launches], ...])."""
    import torch
    from paper_2605_08755_gb300 import _lib
    mp = 1 if wp.M <= 1 else 2 if wp.M <= 2 else 4 if wp.M <= 4 else 8 if wp.M <= 8 else 16
    groups = {}
    for i, (*_, q) in enumerate(wp.linears):
        key = f"gemm_kernel<{q.bits}, {mp}, {wp.configs[i].tiles_per_cta}>"
        groups.setdefault(key, []).append(i)
    rows = []
    for key, idxs in groups.items():
        def run(s=None):
            for i in idxs:
                q = wp.linears[i][3]
                _lib.laq_gemm_wxg128(wp.X[i], q.packed, q.s, q.z, q.bits, Y=wp.Y[i],
                                     config=wp.configs[i], stream=s)
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g, stream=stream):
            run(stream)
        ms = time_graph(g, stream, reps, dev)
        nbytes = sum(wp.linears[i][3].bytes_per_call(wp.M) for i in idxs)
        shapes = {}
        for i in idxs:
            kn = (wp.linears[i][3].K, wp.linears[i][3].N)
            shapes[kn] = shapes.get(kn, 0) + 1
        rows.append((key, len(idxs), nbytes, ms * 1e3, [[k, n, c] for (k, n), c in sorted(shapes.items())]))
        del g
    return rows


VARIANTS = {
    # name: (fused q|k|v and gate|up, one persistent laq_gemm_chain launch)
    "graph_252": (False, False),
    "graph_fused": (True, False),
    "chain_252": (False, True),
    "chain_fused": (True, True),
}


def describe(name, wp):
    fused, chain = VARIANTS[name]
    what = ("252 projections as 144 GEMVs (q|k|v and gate|up over concatenated columns, "
            "identical per-column codes and results)" if fused else "252 GEMVs")
    how = ("one persistent laq_gemm_chain launch (stages q|k|v -> o -> gate|up -> down)"
           if chain else f"{wp.launches} laq_gemm_wxg128 launches in one CUDA graph (PDL)")
    return f"{what}, {how}"


def build_pass(a, dev, name):
    from paper_2605_08755_gb300.weight_pass import WeightPass
    fused, chain = VARIANTS[name]
    chain = chain and a.M <= 4
    if VARIANTS[name][1] and not chain:
        return None
    return WeightPass(model=a.model, bits=a.bits, M=a.M, layers=a.layers,
                      outliers=(a.model == "qwen3-8b"), device=dev, fuse=fused, chain=chain)


def run_laq(a, world, rank, local):
    import torch

    import __graft_entry__

    __graft_entry__.build()
    dev = torch.device("cuda", local)
    torch.cuda.set_device(dev)
    peak, peak_kind = load_peaks()
    stream = torch.cuda.Stream(dev)

    # Every variant of the pass computes the same Y; each is timed briefly, the fastest is
    # the headline and gets the full timed run below.
    variants = {}
    prep_ms = None
    for name in VARIANTS:
        t0 = time.perf_counter()
        wp = build_pass(a, dev, name)
        if wp is None:
            continue
        torch.cuda.synchronize(dev)
        if prep_ms is None:
            prep_ms = (time.perf_counter() - t0) * 1e3
        g = wp.capture(stream=stream)
        ms = min(time_graph(g, stream, max(20, min(a.steps, 300)), dev) for _ in range(2))
        variants[name] = {"launches_per_step": wp.launches, "us_per_step": ms * 1e3,
                          "gbs": wp.bytes_per_pass() / (ms * 1e-3) / 1e9,
                          "what": describe(name, wp)}
        del g, wp
        torch.cuda.empty_cache()
    head = min(variants, key=lambda n: variants[n]["us_per_step"])

    wp = build_pass(a, dev, head)
    bytes_step = wp.bytes_per_pass()
    graph = wp.capture(stream=stream)
    with torch.cuda.stream(stream):
        for _ in range(a.warmup):
            graph.replay()
    torch.cuda.synchronize(dev)

    starts = [torch.cuda.Event(enable_timing=True) for _ in range(a.steps)]
    ends = [torch.cuda.Event(enable_timing=True) for _ in range(a.steps)]
    with ClockSampler(local) as clk:
        barrier(world)
        torch.cuda.synchronize(dev)
        with torch.cuda.stream(stream):
            for i in range(a.steps):
                starts[i].record(stream)
                graph.replay()
                ends[i].record(stream)
        torch.cuda.synchronize(dev)
        barrier(world)
    clocks = clk.summary()
    step_ms = sorted(starts[i].elapsed_time(ends[i]) for i in range(a.steps))
    total_ms = max_over_ranks(world, starts[0].elapsed_time(ends[-1]), dev)
    ms_per_step = total_ms / a.steps
    value = sum_over_ranks(world, bytes_step * a.steps, dev) / (total_ms * 1e-3) / 1e9
    if wp.chain:
        from paper_2605_08755_gb300 import chain_status
        if chain_status(wp.ws) != 0:
            raise RuntimeError("laq_gemm_chain reported a device-side error")

    # The dominant kernel: the chain kernel itself, or the GEMV instance of the graph with the
    # most device time (per-instance graphs of the step's launches, timed on their stream).
    if wp.chain:
        rows = [("chain_kernel<%d, %d>" % (a.bits, 1 if a.M <= 1 else 2 if a.M <= 2 else 4),
                 1, bytes_step, ms_per_step * 1e3, None)]
    else:
        rows = kernel_breakdown(wp, stream, dev)
    dom = max(rows, key=lambda r: r[3])
    kernel_gbs = dom[2] / (dom[3] * 1e-6) / 1e9

    # End to end through the public API with host buffers: every step copies all of its X
    # from pinned host memory, runs the pass and copies all of its Y back, as a serving loop
    # would: double-buffered, the next step's X travels on a copy stream while this step's pass
    # runs, and this step's Y (first copied aside on the device) returns while the next pass
    # runs.  Every copy of every step lies inside the timed region (the main stream joins the
    # copy stream before the end event).
    xh = torch.empty(wp.Xbuf.shape, dtype=wp.Xbuf.dtype, pin_memory=True)
    xh.copy_(wp.Xbuf)
    yh = [torch.empty(wp.Ybuf.shape, dtype=wp.Ybuf.dtype, pin_memory=True) for _ in range(2)]
    xd = [torch.empty_like(wp.Xbuf) for _ in range(2)]   # landing buffers of the H2D copies
    yd = [torch.empty_like(wp.Ybuf) for _ in range(2)]   # Y set aside for the D2H copies
    copy = torch.cuda.Stream(dev)
    ev = lambda: torch.cuda.Event()  # noqa: E731
    x_in, x_free, y_out, y_free = ([ev(), ev()] for _ in range(4))
    e2e_steps = max(10, min(a.steps, 400))
    torch.cuda.synchronize(dev)
    e_a, e_b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e_a.record(stream)
    copy.wait_stream(stream)
    with torch.cuda.stream(copy):
        xd[0].copy_(xh, non_blocking=True)
        x_in[0].record(copy)
    for t in range(e2e_steps):
        b = t % 2
        with torch.cuda.stream(stream):
            stream.wait_event(x_in[b])              # this step's X has arrived
            wp.Xbuf.copy_(xd[b])
            x_free[b].record(stream)
        if t + 1 < e2e_steps:                       # the next step's X, during this pass
            with torch.cuda.stream(copy):
                copy.wait_event(x_free[1 - b])
                xd[1 - b].copy_(xh, non_blocking=True)
                x_in[1 - b].record(copy)
        with torch.cuda.stream(stream):
            graph.replay()
            if t >= 2:
                stream.wait_event(y_free[b])        # yd[b] of step t - 2 has left
            yd[b].copy_(wp.Ybuf)
            y_out[b].record(stream)
        with torch.cuda.stream(copy):               # this step's Y, during the next pass
            copy.wait_event(y_out[b])
            yh[b].copy_(yd[b], non_blocking=True)
            y_free[b].record(copy)
    stream.wait_stream(copy)
    e_b.record(stream)
    torch.cuda.synchronize(dev)
    e2e_ms = max_over_ranks(world, e_a.elapsed_time(e_b), dev) / e2e_steps
    e2e_gbs = sum_over_ranks(world, bytes_step, dev) / (e2e_ms * 1e-3) / 1e9
    h2d, d2h = wp.Xbuf.numel() * 2, wp.Ybuf.numel() * 2
    launches = wp.launches
    del graph, wp
    torch.cuda.empty_cache()

    fp16_us = None
    if not a.no_fp16 and rank == 0:
        fp16_us, _ = fp16_context(a, dev)

    cpu = None
    if rank == 0:
        smp = OracleSample(a.model, a.bits, a.M)
        b, spent, names = smp.run(a.cpu_seconds)
        cpu = {"value": b / spent / 1e9, "unit": "GB/s", "cores": 1, "kind": "oracle",
               "sample": f"C oracle (fp64, one thread) dequantize-and-multiply of "
                         f"{len(names)} whole projections of layer 0, round-robin over "
                         f"q,k,v,o,gate,up,down, {spent:.1f} s of CPU work; quantization not "
                         f"timed"}

    if rank != 0:
        return
    pct = lambda q: step_ms[min(len(step_ms) - 1, int(q * (len(step_ms) - 1)))]
    line = {
        "metric": METRIC, "value": value, "unit": "GB/s", "n_gpus": world, "steps": a.steps,
        "warmup": a.warmup, "ms_per_step": ms_per_step, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None,
        "dtype": f"u{a.bits} codes + fp16 (fp32 accumulate)", "data": "synthetic",
        "config": {"workload": workload_name(a) + ": " + variants[head]["what"],
                   "model": a.model, "bits": a.bits, "M": a.M, "pass_variant": head,
                   "launches_per_step": launches, "bytes_per_step": bytes_step,
                   "us_per_step": ms_per_step * 1e3,
                   "pct_of_peak": 100.0 * value / world / peak,
                   "peak_gbs": peak, "peak_kind": peak_kind,
                   "l2": "inputs larger than L2 (packed weights per step >> 129 MB)",
                   "step_ms_p10_p50_p90": [pct(0.1), pct(0.5), pct(0.9)],
                   "prep_ms": prep_ms,
                   "variants_us_per_step": {k: round(v["us_per_step"], 1)
                                            for k, v in variants.items()},
                   "variants_gbs": {k: round(v["gbs"], 1) for k, v in variants.items()},
                   "fp16_torch_matmul_us_per_step": fp16_us,
                   "speedup_vs_fp16_torch": (fp16_us / (ms_per_step * 1e3)) if fp16_us else None,
                   "parallelism": f"replicas x{world}"},
        "roofline": {"bound": "hbm", "achieved": kernel_gbs, "peak": peak, "unit": "GB/s",
                     "frac": kernel_gbs / peak, "traffic": traffic_for(dom[0], a, head, dom[4]),
                     "kernel": dom[0], "launches_per_step": dom[1],
                     "us_per_launch": dom[3] / dom[1], "bytes_per_launch": dom[2] / dom[1],
                     "peak_kind": peak_kind,
                     "instances": [{"kernel": k, "launches": n, "us_per_step": us,
                                    "gbs": nb / (us * 1e-6) / 1e9, "shapes": sh}
                                   for k, n, nb, us, sh in rows]},
        "cpu_baseline": cpu,
        "e2e": {"value": e2e_gbs, "unit": "GB/s", "h2d_bytes_per_step": h2d,
                "d2h_bytes_per_step": d2h, "us_per_step": e2e_ms * 1e3},
        "gpu_launches": launches * a.steps,
        "clocks": clocks,
    }
    print(json.dumps(line), flush=True)


def main():
    a = parse()
    world, rank, local = dist_setup(a)
    if a.impl == "reference":
        run_reference(a, world, rank)
    else:
        run_laq(a, world, rank, local)
    if world > 1:
        import torch.distributed as dist
        dist.destroy_process_group()


if __name__ == "__main__":
    main()
