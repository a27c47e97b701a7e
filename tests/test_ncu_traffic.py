"""The ncu launch-list summariser behind bench.py's roofline.traffic (host logic, no GPU)."""
import json
import subprocess
import sys

import pytest

from paper_2605_08755_gb300 import ncu_traffic
from paper_2605_08755_gb300.weight_pass import pass_plan

HEADER = ('"ID","Process ID","Process Name","Host Name","Kernel Name","Context","Stream",'
          '"Block Size","Grid Size","Device","CC","Section Name","Metric Name","Metric Unit",'
          '"Metric Value"\n')


def fake_csv(path, kernels, nbytes, flag="false"):
    rows = ["==PROF== Connected to process 1\n", HEADER]
    for i, (k, b) in enumerate(zip(kernels, nbytes)):
        name = (f"void laq::(anonymous namespace)::gemm_kernel<(int){k[0]}, (int){k[1]}, "
                f"(int){k[2]}, {flag}>(laq::(anonymous namespace)::Params)")
        for metric, unit, val in (("dram__bytes_read.sum", "Mbyte", f"{b / 1e6:.3f}"),
                                  ("dram__bytes_write.sum", "byte", "1,000"),
                                  ("gpu__time_duration.sum", "ns", "5000")):
            rows.append(f'"{i}","1","python","h","{name}","1","7","(256, 1, 1)","(152, 1, 1)",'
                        f'"0","10.3","Command line profiler metrics","{metric}","{unit}","{val}"\n')
    path.write_text("".join(rows))


@pytest.mark.parametrize("flag", ["false", "(bool)0"])
def test_groups_launches_by_instance_and_projection_shapes(tmp_path, flag):
    plan = pass_plan("qwen3-4b", True, 2)  # q|k|v, o, gate|up, down per layer
    kernels = [(3, 1, 2), (3, 1, 1), (3, 1, 4), (3, 1, 2)] * 2
    nbytes = [6.3e6, 4.2e6, 19.9e6, 9.9e6] * 2
    csvp = tmp_path / "l.csv"
    fake_csv(csvp, kernels, nbytes, flag)
    launches = ncu_traffic.read_launches(str(csvp))
    assert [k for k, _, _ in launches] == [f"gemm_kernel<{a}, {b}, {c}>" for a, b, c in kernels]
    assert launches[0][1] == pytest.approx(6.3e6 + 1000)
    out = tmp_path / "t.json"
    r = subprocess.run([sys.executable, "-m", "paper_2605_08755_gb300.ncu_traffic", str(csvp),
                        "--variant", "graph_fused", "--layers", "2", "--write", str(out)],
                       capture_output=True, text=True, check=True)
    assert "gemm_kernel<3, 1, 2> (qkv, down) | 4 |" in r.stdout
    t = json.loads(out.read_text())
    e = t["gemm_kernel<3, 1, 2> qwen3-4b W3 M=1 graph_fused"]
    assert e["launches"] == 4
    assert e["dram_bytes_per_launch"] == round((6.3e6 + 9.9e6) / 2 + 1000, -3)
    K_N = sorted({(K, N) for *_, name, K, N in plan if name in ("qkv", "down")})
    assert e["shapes"] == [[K, N, 2] for K, N in K_N]
    assert e["sources_sha256"] == ncu_traffic.sources_sha256()


def test_rejects_a_log_that_is_not_one_pass(tmp_path):
    csvp = tmp_path / "l.csv"
    fake_csv(csvp, [(3, 1, 2)] * 3, [1e6] * 3)
    r = subprocess.run([sys.executable, "-m", "paper_2605_08755_gb300.ncu_traffic", str(csvp),
                        "--variant", "graph_fused", "--layers", "1"], capture_output=True, text=True)
    assert r.returncode != 0 and "3 launches" in (r.stderr + r.stdout)


@pytest.mark.parametrize("flag", ["true", "(bool)1"])
def test_prologue_instances_are_named_apart(tmp_path, flag):
    csvp = tmp_path / "l.csv"
    fake_csv(csvp, [(3, 1, 2)], [1e6], flag)
    assert ncu_traffic.read_launches(str(csvp))[0][0] == "gemm_kernel<3, 1, 2> prologue"
