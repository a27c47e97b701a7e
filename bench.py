"""Benchmark: the Qwen3-shaped decode-step weight pass (W3G128 by default) on GB300.

One step = one replay of a CUDA graph holding every quantized projection of the model once
(36 layers x q, k, v, o, gate, up, down, M = 1), i.e. the weight streaming of one batch-1
decode step.  The pass has equivalent forms (252 ``laq_gemm_wxg128`` launches; 144 with q|k|v
and gate|up fused over concatenated columns; one persistent ``laq_pass_run`` launch over per-SM
weight streams); each is timed briefly and the fastest gets the full timed run.  Quantization
and packing (``laq_quantize_rtn``, ``laq_pack``) are the offline model-preparation steps and run
once before timing; their time is reported as ``prep_ms``.  Synthetic weights ~ N(0, 0.02^2)
and activations ~ N(0, 1) stand in for the paper's Qwen3 checkpoints.

Prints one JSON line.  ``value`` is the achieved HBM bandwidth of the pass (algorithmic bytes =
packed codes + s + z + X + Y, per step, all ranks) over the device time of the timed replays.
Unless ``--no-sweep``, the line also carries ``sweep``: the other measured workloads (one
1024 x 1024 GEMV, each projection of a Qwen3-4B layer, the Qwen3-4B pass at W3 and W4 for
M = 1, 2, 4, 8, 16, the Qwen3-8B pass with outliers at M = 1 and 16, and a whole decode step
with and without an online rotation), each timed on its own after the headline.

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
    ap.add_argument("--no-sweep", action="store_true", help="skip the other workloads")
    ap.add_argument("--variant", default=None, choices=["graph_252", "graph_fused", "planned_fused"],
                    help="time only this form of the pass (for profiling runs, where the "
                         "profiler's serialised launches would change which form is fastest)")
    ap.add_argument("--cpu-seconds", type=float, default=12.0,
                    help="CPU work budget of the oracle baseline sample")
    return ap.parse_args()


def workload_name(a):
    return (f"{a.model} decode-step weight pass, {a.layers} layers x 7 projections, "
            f"W{a.bits}G128, M={a.M}")


def workload_config(a):
    """The ``config`` of both arms: the same workload."""
    return {"workload": workload_name(a), "bits": a.bits, "M": a.M, "layers": a.layers,
            "shapes": a.model,
            "l2": "inputs larger than L2 (packed weights per step >> 129 MB)"}


def host_cpu():
    """(CPU model name, cores available to this process)."""
    name = None
    try:
        with open("/proc/cpuinfo") as f:
            for line in f:
                k, _, v = line.partition(":")
                if k.strip() in ("model name", "Model Name", "CPU part") and v.strip():
                    name = v.strip()
                    if k.strip() != "CPU part":
                        break
    except OSError:
        pass
    if name is None or name.startswith("0x"):
        try:
            out = subprocess.run(["lscpu"], capture_output=True, text=True, timeout=10).stdout
            for line in out.splitlines():
                if line.split(":")[0].strip() == "Model name":
                    name = line.split(":", 1)[1].strip()
                    break
        except (OSError, subprocess.SubprocessError):
            pass
    return name or "unknown", len(os.sched_getaffinity(0))


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
    column slice of one, when a short step is asked for); ``run_quantize`` times its quantizer
    and packer, the offline step, separately."""

    def __init__(self, model, bits, M, seed=0):
        from oracle import c_oracle
        from paper_2605_08755_gb300 import inputs
        from paper_2605_08755_gb300.weight_pass import shapes
        self.co = c_oracle
        self.bits, self.M = bits, M
        self.items = []
        self.weights = []
        for pi, (name, K, N) in enumerate(shapes(model)):
            sd = inputs.proj_seed(seed, 0, pi)
            W = inputs.weights(K, N, sd, outliers=(model == "qwen3-8b"))
            codes, s, z = c_oracle.quantize_rtn_threads(W, bits)
            self.items.append((f"L0.{name}", codes, s, z, inputs.activations(M, K, sd)))
            self.weights.append((f"L0.{name}", W))
        self.next = 0

    def run_quantize(self, seconds, threaded=True):
        """The oracle's RTN quantizer (``threaded``: over the host's threads) and its packer on
        whole layer-0 projections, round-robin, for about ``seconds``; returns (weights,
        quantize seconds, pack seconds, projections)."""
        n = qs = ps = 0.0
        names = []
        i = 0
        while True:
            name, W = self.weights[i % len(self.weights)]
            i += 1
            t0 = time.perf_counter()
            codes, _, _ = (self.co.quantize_rtn_threads if threaded else self.co.quantize_rtn)(
                W, self.bits)
            t1 = time.perf_counter()
            self.co.pack(codes, self.bits)
            t2 = time.perf_counter()
            qs += t1 - t0
            ps += t2 - t1
            n += W.size
            names.append(name)
            if qs + ps >= seconds:
                break
        return n, qs, ps, names

    def nbytes(self, K, N):
        return K * N * self.bits // 8 + (K // 128) * N * 3 + 2 * self.M * K + 2 * self.M * N

    def run(self, seconds, max_cols=None, threaded=False):
        """Oracle work for about ``seconds`` (``threaded``: the all-cores GEMM, its output
        columns split over the host's threads); returns (bytes, seconds spent, items done)."""
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
            (self.co.gemm_threads if threaded else self.co.gemm)(X, codes, s, z)
            spent += time.perf_counter() - t0
            done += self.nbytes(K, N)
            names.append(name)
            if spent >= seconds:
                break
        return done, spent, names


def oracle_single_linear(bits, reps=20):
    """The oracle, one thread, on a single 1024 x 1024 W{bits}G128 linear at M = 1 (the shapes
    and distributions of the GPU's gemv_1024 sweep entry): median time of its
    dequantize-and-multiply over ``reps`` calls."""
    from oracle import c_oracle
    from paper_2605_08755_gb300 import inputs
    W = inputs.weights(1024, 1024, 0)
    codes, s, z = c_oracle.quantize_rtn(W, bits)
    X = inputs.activations(1, 1024, 0)
    ts = []
    for _ in range(reps):
        t0 = time.perf_counter()
        c_oracle.gemm(X, codes, s, z)
        ts.append(time.perf_counter() - t0)
    us = 1e6 * statistics.median(ts)
    nbytes = 1024 * 1024 * bits // 8 + 8 * 1024 * 3 + 2 * 1024 + 2 * 1024
    return {"us_per_gemv": us, "gbs": nbytes / us / 1e3, "threads": 1}


# ------------------------------------------------------------------ reference arm


def run_reference(a, world, rank):
    """The oracle, as it stands, on the host cores (its all-cores GEMM): each step is a bounded
    sample of the pass (a column slice of one layer-0 projection, sized so the whole run stays
    within a few minutes)."""
    if rank != 0:
        return
    smp = OracleSample(a.model, a.bits, a.M)
    cpu_name, avail = host_cpu()
    per_step_s = min(0.25, max(0.002, 90.0 / max(1, a.steps + a.warmup)))
    # calibrate columns per step on the first projection
    name, codes, *_ = smp.items[0]
    K, N = codes.shape
    b, sp, _ = smp.run(0.0, max_cols=256, threaded=True)
    cols = int(max(64, min(N, 256 * per_step_s / max(sp, 1e-6))) // 64 * 64)
    smp.next = 0
    for _ in range(a.warmup):
        smp.run(0.0, max_cols=cols, threaded=True)
    tot_b, tot_s, names = 0, 0.0, []
    step_s = []
    for _ in range(a.steps):
        b, sp, nm = smp.run(0.0, max_cols=cols, threaded=True)
        tot_b += b
        tot_s += sp
        step_s.append(sp)
        names += nm
    value = tot_b / tot_s / 1e9
    threads = smp.co.threads()
    sample = (f"C oracle (fp64) dequantize-and-multiply, output columns split over {threads} "
              f"threads; each step = the first {cols} columns of one layer-0 projection, "
              f"round-robin over q,k,v,o,gate,up,down; {tot_s:.3g} s of CPU work over "
              f"{a.steps} steps; quantization not timed; host CPU {cpu_name}, {avail} cores "
              f"available")
    line = {"metric": METRIC, "value": value, "unit": "GB/s", "n_gpus": a.gpus,
            "steps": a.steps, "warmup": a.warmup,
            "ms_per_step": 1e3 * statistics.median(step_s), "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
            "impl": "reference", "config": workload_config(a),
            "cpu_baseline": {"value": value, "unit": "GB/s", "cores": threads, "kind": "oracle",
                             "cpu": cpu_name, "sample": sample},
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
    # name: (fused q|k|v and gate|up, form): "graph" = one laq_gemm_wxg128 launch per GEMV in a
    # CUDA graph (PDL), "planned" = one persistent laq_pass_run launch (M <= 4)
    "graph_252": (False, "graph"),
    "graph_fused": (True, "graph"),
    "planned_fused": (True, "planned"),
}


def describe(name, wp):
    fused, form = VARIANTS[name]
    what = ("252 projections as 144 GEMVs (q|k|v and gate|up over concatenated columns, "
            "identical per-column codes and results)" if fused else "252 GEMVs")
    how = ("one persistent laq_pass_run launch over per-SM weight streams (stages q|k|v -> o -> "
           "gate|up -> down)" if form == "planned"
           else f"{wp.launches} laq_gemm_wxg128 launches in one CUDA graph (PDL)")
    return f"{what}, {how}"


def build_pass(a, dev, name, model=None, bits=None, M=None):
    from paper_2605_08755_gb300.weight_pass import WeightPass
    model = model or a.model
    bits = bits or a.bits
    M = M or a.M
    fused, form = VARIANTS[name]
    if form == "planned" and M > 4:
        return None
    return WeightPass(model=model, bits=bits, M=M, layers=a.layers,
                      outliers=(model == "qwen3-8b"), device=dev, fuse=fused,
                      planned=(form == "planned"))


def pass_status_ok(wp):
    return wp.plan.status() == 0 if wp.planned else True


# ------------------------------------------------------------------ the other workloads


def sweep_gemv_1024(a, dev, stream):
    """One 1024 x 1024 W3G128 GEMV at M = 1 (421,888 algorithmic bytes, L2-resident on its
    own): timed over 640 distinct copies (270 MB, more than twice L2) launched back to back in
    one CUDA graph, so each launch reads its weights from HBM."""
    import torch

    from paper_2605_08755_gb300 import _lib, inputs
    K = N = 1024
    copies = 640
    W = inputs.weights_torch(K, N, 1, dev)
    codes, s_, z_ = _lib.laq_quantize_rtn(W, 3)
    packed = _lib.laq_pack(codes, 3)
    P = packed.repeat(copies).view(copies, -1)
    S = s_.repeat(copies, 1).view(copies, *s_.shape)
    Z = z_.repeat(copies, 1).view(copies, *z_.shape)
    X = inputs.activations_torch(1, K, 1, dev)
    Y = torch.empty((copies, 1, N), dtype=torch.float16, device=dev)
    cfg = _lib.laq_gemm_plan(1, K, N, 3, torch.cuda.get_device_properties(dev).multi_processor_count)
    cfg.pdl = 1

    def run(st=None):
        for i in range(copies):
            _lib.laq_gemm_wxg128(X, P[i], S[i], Z[i], 3, Y=Y[i], config=cfg, stream=st)
    run()
    torch.cuda.synchronize(dev)
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, stream=stream):
        run(stream)
    ms = min(time_graph(g, stream, 20, dev) for _ in range(2))
    us = ms * 1e3 / copies
    nbytes = K * N * 3 // 8 + (K // 128) * N * 3 + 2 * K + 2 * N
    del g, P, S, Z, Y
    return {"us_per_gemv": us, "gbs": nbytes / (us * 1e-6) / 1e9, "bytes_per_gemv": nbytes,
            "l2": f"{copies} distinct copies per replay ({copies * nbytes / 1e6:.0f} MB)",
            "launch": "back to back in one CUDA graph, PDL"}


def sweep_layer_projections(a, dev, stream):
    """Each projection of a Qwen3-4B layer (W3G128, M = 1): a CUDA graph of that projection's
    36 launches of the 36-layer pass (36 distinct weights, HBM-cold), µs per GEMV."""
    import torch

    from paper_2605_08755_gb300 import _lib
    wp = build_pass(a, dev, "graph_252", model="qwen3-4b", bits=3, M=1)
    out = {}
    for name in ("q", "k", "v", "o", "gate", "up", "down"):
        idx = [i for i, (_, _, nm, _) in enumerate(wp.linears) if nm == name]

        def run(st=None, idx=idx):
            for i in idx:
                q = wp.linears[i][3]
                _lib.laq_gemm_wxg128(wp.X[i], q.packed, q.s, q.z, q.bits, Y=wp.Y[i],
                                     config=wp.configs[i], stream=st)
        run()
        torch.cuda.synchronize(dev)
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g, stream=stream):
            run(stream)
        ms = min(time_graph(g, stream, 50, dev) for _ in range(2))
        us = ms * 1e3 / len(idx)
        q = wp.linears[idx[0]][3]
        nb = q.bytes_per_call(1)
        out[name] = {"K": q.K, "N": q.N, "us_per_gemv": us, "gbs": nb / (us * 1e-6) / 1e9}
        del g
    del wp
    torch.cuda.empty_cache()
    return out


def sweep_pass(a, dev, stream, model, bits, M, variants):
    """A whole decode-step weight pass in each form of ``variants``: µs per pass and GB/s."""
    import torch
    res = {}
    for name in variants:
        wp = build_pass(a, dev, name, model=model, bits=bits, M=M)
        if wp is None:
            continue
        g = wp.capture(stream=stream)
        ms = min(time_graph(g, stream, 30, dev) for _ in range(2))
        if not pass_status_ok(wp):
            raise RuntimeError(f"{name}: device-side error")
        res[name] = {"us_per_pass": ms * 1e3,
                     "gbs": wp.bytes_per_pass() / (ms * 1e-3) / 1e9}
        del g, wp
        torch.cuda.empty_cache()
    best = min(res, key=lambda n: res[n]["us_per_pass"])
    return {"best": best, "us_per_pass": res[best]["us_per_pass"], "gbs": res[best]["gbs"],
            "variants": res}


def sweep_decode_step(a, dev, stream, rounds):
    """A whole Qwen3-4B decode step (W3G128, M = 1, context 2048) on the library's kernels, and
    the same step with an online pairwise rotation of ``rounds`` rounds before every projection
    (the rotation-based comparison): µs and tokens per second."""
    import torch

    from paper_2605_08755_gb300.decode_case import time_graph as tg
    from paper_2605_08755_gb300.decode_step import DecodeStep
    out = {}
    for label, rot in (("laquant", 0), (f"rotated_{rounds}_rounds", rounds)):
        st = DecodeStep(model="qwen3-4b", bits=3, M=1, context=2048, rotation_rounds=rot)
        g = st.capture(stream=stream)
        us = tg(g, stream, 30)
        out[label] = {"us_per_token": us, "tokens_per_s": 1e6 / us, "launches": st.launches}
        del g, st
        torch.cuda.empty_cache()
    out["faster_without_rotation"] = (out[f"rotated_{rounds}_rounds"]["us_per_token"]
                                      / out["laquant"]["us_per_token"] - 1.0)
    return out


def run_sweep(a, dev, stream):
    """The workloads besides the headline, each on its own; a failing item records its error."""
    sweep = {}
    items = [
        ("gemv_1024x1024_w3_m1", lambda: sweep_gemv_1024(a, dev, stream)),
        ("qwen3_4b_layer_w3_m1_per_projection", lambda: sweep_layer_projections(a, dev, stream)),
    ]
    for bits in (3, 4):
        for M in (1, 2, 4, 8, 16):
            items.append((f"qwen3_4b_pass_w{bits}_m{M}",
                          lambda bits=bits, M=M: sweep_pass(
                              a, dev, stream, "qwen3-4b", bits, M,
                              ["graph_fused", "planned_fused"])))
    for M in (1, 16):
        items.append((f"qwen3_8b_outliers_pass_w3_m{M}",
                      lambda M=M: sweep_pass(a, dev, stream, "qwen3-8b", 3, M,
                                             ["graph_fused", "planned_fused"])))
    items.append(("qwen3_4b_decode_step_w3_m1", lambda: sweep_decode_step(a, dev, stream, 8)))
    t_all = time.perf_counter()
    for name, fn in items:
        t0 = time.perf_counter()
        try:
            sweep[name] = fn()
        except Exception as e:  # noqa: BLE001 - recorded, the headline stands
            sweep[name] = {"error": f"{type(e).__name__}: {e}"[:300]}
        sweep[name]["wall_s"] = round(time.perf_counter() - t0, 2)
    sweep["wall_s"] = round(time.perf_counter() - t_all, 2)
    return sweep


# ------------------------------------------------------------------ the headline


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
    for name in ([a.variant] if a.variant else VARIANTS):
        t0 = time.perf_counter()
        wp = build_pass(a, dev, name)
        if wp is None:
            continue
        torch.cuda.synchronize(dev)
        if prep_ms is None:
            prep_ms = (time.perf_counter() - t0) * 1e3
        g = wp.capture(stream=stream)
        ms = min(time_graph(g, stream, max(20, min(a.steps, 300)), dev) for _ in range(2))
        if not pass_status_ok(wp):
            raise RuntimeError(f"{name}: laq_pass_run reported a device-side error")
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
    if not pass_status_ok(wp):
        raise RuntimeError("laq_pass_run reported a device-side error")

    # The dominant kernel: the persistent pass kernel itself, or the GEMV instance of the graph
    # with the most device time (per-instance graphs of the step's launches, timed on their
    # stream).
    if wp.planned:
        mp = 1 if a.M <= 1 else 2 if a.M <= 2 else 4
        rows = [(f"pass_kernel<{a.bits}, {mp}>", 1, bytes_step, ms_per_step * 1e3, None)]
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
    if not pass_status_ok(wp):
        raise RuntimeError("laq_pass_run reported a device-side error")
    e2e_ms = max_over_ranks(world, e_a.elapsed_time(e_b), dev) / e2e_steps
    e2e_gbs = sum_over_ranks(world, bytes_step, dev) / (e2e_ms * 1e-3) / 1e9
    h2d, d2h = wp.Xbuf.numel() * 2, wp.Ybuf.numel() * 2
    launches = wp.launches
    del graph, wp
    torch.cuda.empty_cache()

    fp16_us = None
    if not a.no_fp16 and rank == 0:
        fp16_us, _ = fp16_context(a, dev)

    sweep = None
    if not a.no_sweep and rank == 0:
        sweep = run_sweep(a, dev, stream)

    cpu = None
    if rank == 0:
        smp = OracleSample(a.model, a.bits, a.M)
        cpu_name, avail = host_cpu()
        b1, s1, n1 = smp.run(min(4.0, a.cpu_seconds / 3))
        smp.next = 0
        b, spent, names = smp.run(a.cpu_seconds, threaded=True)
        threads = smp.co.threads()
        cpu = {"value": b / spent / 1e9, "unit": "GB/s", "cores": threads, "kind": "oracle",
               "cpu": cpu_name, "cores_available": avail,
               "single_thread_value": b1 / s1 / 1e9,
               "sample": f"C oracle (fp64) dequantize-and-multiply, output columns split over "
                         f"{threads} threads, of {len(names)} whole projections of layer 0, "
                         f"round-robin over q,k,v,o,gate,up,down, {spent:.1f} s of wall time "
                         f"(single-threaded: {len(n1)} projections in {s1:.1f} s); the "
                         f"quantizer and packer timed separately (quantize_pack)"}
        cpu["single_linear_1024"] = oracle_single_linear(a.bits)
        nw, qs, ps, qn = smp.run_quantize(min(4.0, a.cpu_seconds / 3))
        cpu["quantize_pack"] = {
            "quantize_weights_per_s": nw / qs, "pack_weights_per_s": nw / ps,
            "sample": f"oracle RTN quantizer (fp64, columns split over {threads} threads) and "
                      f"packer (one thread) on {len(qn)} whole layer-0 projections "
                      f"({nw / 1e6:.0f} M weights): {qs:.2f} s quantizing, {ps:.2f} s packing"}

    if rank != 0:
        return
    pct = lambda q: step_ms[min(len(step_ms) - 1, int(q * (len(step_ms) - 1)))]
    line = {
        "metric": METRIC, "value": value, "unit": "GB/s", "n_gpus": world, "steps": a.steps,
        "warmup": a.warmup, "ms_per_step": ms_per_step, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None,
        "dtype": f"u{a.bits} codes + fp16 (fp32 accumulate)", "data": "synthetic",
        "config": workload_config(a),
        "details": {"pass_variant": head, "what": variants[head]["what"],
                    "launches_per_step": launches, "bytes_per_step": bytes_step,
                    "us_per_step": ms_per_step * 1e3,
                    "pct_of_peak": 100.0 * value / world / peak,
                    "peak_gbs": peak, "peak_kind": peak_kind,
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
        "sweep": sweep,
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
