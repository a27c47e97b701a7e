"""Per-instance DRAM traffic of a decode-step pass from an ncu launch list.

    python -m paper_2605_08755_gb300.ncu_traffic launches_graph_fused.csv \\
        --variant graph_fused [--model qwen3-4b --bits 3 --M 1] [--write profiles/traffic.json]

The CSV is ncu's ``--csv`` log of ``--metrics dram__bytes_read.sum,dram__bytes_write.sum,
gpu__time_duration.sum`` over exactly one step's GEMV launches of a graph form (selected with
``pass_case``'s ``-s L -c L``), so launch i is the pass's i-th GEMV.  Launches are grouped by
kernel instance (its template arguments, as ``bench.py`` names them); each group's entry holds
the DRAM bytes per launch, the projection shapes it ran and the sha256 of the kernel's sources,
so that ``bench.py`` reports the figure only for the same kernel and launch mix.  Prints a
markdown table of the groups.
"""
import argparse
import csv
import hashlib
import json
import os
import re

from .weight_pass import pass_plan
from . import inputs

SOURCES = ["laq_gemm_kernel.cuh", "laq_gemm.cu", "laq_device.cuh"]
CSRC = os.path.join(os.path.dirname(os.path.abspath(__file__)), "csrc")


def sources_sha256():
    h = hashlib.sha256()
    for name in SOURCES:
        with open(os.path.join(CSRC, name), "rb") as f:
            h.update(f.read())
    return h.hexdigest()


def read_launches(path):
    """[(kernel instance, dram bytes, duration us)] in launch order."""
    with open(path, newline="") as f:
        lines = [ln for ln in f if ln.startswith('"')]  # ncu prefixes its own messages with ==
    launches = {}
    for row in csv.DictReader(lines):
        lid = int(row["ID"])
        m = re.search(r"gemm_kernel<([^>]*)>", row["Kernel Name"])
        if not m:
            continue
        # <BITS, MP, NT, PRO>: ncu writes the ints as (int)3 and the flag as false/true or
        # (bool)0/1; the prologue instances get their own name
        targs = [t.strip() for t in re.sub(r"\([a-z ]+\)", "", m.group(1)).split(",")]
        pro = len(targs) > 3 and targs[3] in ("true", "1")
        name = "gemm_kernel<" + ", ".join(targs[:3]) + ">" + (" prologue" if pro else "")
        d = launches.setdefault(lid, {"kernel": name})
        val = float(row["Metric Value"].replace(",", ""))
        unit = row["Metric Unit"]
        scale = {"byte": 1, "Kbyte": 1e3, "Mbyte": 1e6, "Gbyte": 1e9, "ns": 1e-3, "nsecond": 1e-3,
                 "us": 1.0, "usecond": 1.0, "ms": 1e3, "msecond": 1e3}[unit]
        d[row["Metric Name"]] = val * scale
    return [(d["kernel"], d["dram__bytes_read.sum"] + d["dram__bytes_write.sum"],
             d["gpu__time_duration.sum"]) for _, d in sorted(launches.items())]


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("csv")
    ap.add_argument("--variant", required=True, choices=["graph_252", "graph_fused"])
    ap.add_argument("--model", default="qwen3-4b", choices=["qwen3-4b", "qwen3-8b"])
    ap.add_argument("--bits", type=int, default=3)
    ap.add_argument("--M", type=int, default=1)
    ap.add_argument("--layers", type=int, default=inputs.LAYERS)
    ap.add_argument("--write", default=None, help="traffic table (JSON) to update")
    a = ap.parse_args()
    plan = pass_plan(a.model, a.variant == "graph_fused", a.layers)
    launches = read_launches(a.csv)
    if len(launches) != len(plan):
        raise SystemExit(f"{len(launches)} launches in the log, the pass has {len(plan)}")
    groups = {}
    for (kernel, nbytes, us), (_, _, name, K, N) in zip(launches, plan):
        g = groups.setdefault(kernel, {"bytes": 0.0, "us": 0.0, "n": 0, "shapes": {}, "names": []})
        g["bytes"] += nbytes
        g["us"] += us
        g["n"] += 1
        g["shapes"][(K, N)] = g["shapes"].get((K, N), 0) + 1
        if name not in g["names"]:
            g["names"].append(name)
    total_us = sum(g["us"] for g in groups.values())
    print("| kernel instance (projections) | launches | total (us) | share | DRAM bytes / launch |")
    print("|---|---|---|---|---|")
    for k, g in sorted(groups.items(), key=lambda kv: -kv[1]["us"]):
        print(f"| {k} ({', '.join(g['names'])}) | {g['n']} | {g['us']:.1f} | "
              f"{100 * g['us'] / total_us:.1f} % | {g['bytes'] / g['n'] / 1e6:.3f} MB |")
    if a.write:
        table = {}
        if os.path.exists(a.write):
            with open(a.write) as f:
                table = json.load(f)
        sha = sources_sha256()
        prefix = f" {a.model} W{a.bits} M={a.M} {a.variant}"
        for key in [k for k in table if k.endswith(prefix)]:
            del table[key]
        for k, g in groups.items():
            table[k + prefix] = {
                "dram_bytes_per_launch": int(round(g["bytes"] / g["n"], -3)),
                "launches": g["n"],
                "shapes": [[K, N, c] for (K, N), c in sorted(g["shapes"].items())],
                "sources": SOURCES,
                "sources_sha256": sha,
            }
        with open(a.write, "w") as f:
            json.dump(table, f, indent=1)
            f.write("\n")


if __name__ == "__main__":
    main()
