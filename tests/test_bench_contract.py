"""The bench's JSON line, checked on the host: the reference arm (the oracle
timed on the host cores) on the tiny configuration, run as the driver runs it,
and the kernel byte model that the roofline divides by."""
import json
import os
import subprocess
import sys

import pytest

from tests.conftest import ROOT


def _run_bench(*args):
    env = dict(os.environ, CUDA_VISIBLE_DEVICES="")
    r = subprocess.run([sys.executable, os.path.join(ROOT, "bench.py"), *args], cwd=ROOT, env=env,
                       capture_output=True, text=True, timeout=600)
    assert r.returncode == 0, r.stderr[-2000:]
    lines = [l for l in r.stdout.splitlines() if l.startswith("{")]
    assert len(lines) == 1, r.stdout[-2000:]
    return json.loads(lines[0])


def test_reference_arm_line():
    d = _run_bench("--impl", "reference", "--config", "tiny", "--steps", "2", "--warmup", "1")
    for k in ("metric", "value", "unit", "n_gpus", "steps", "warmup", "ms_per_step", "higher_is_better", "scaling",
              "vs_baseline", "dtype", "data", "config", "impl", "cpu_baseline", "e2e"):
        assert k in d, k
    assert d["impl"] == "reference" and d["steps"] == 2 and d["warmup"] == 1 and d["n_gpus"] == 1
    assert d["unit"] == "tokens/s" and d["higher_is_better"] is True and d["value"] > 0
    assert d["config"]["workload"] == "tiny-shaped fingerprint"
    cb = d["cpu_baseline"]
    assert cb["kind"] == "oracle" and cb["cores"] >= 1 and cb["value"] == d["value"] and "2 timed steps" in cb["sample"]
    e = d["e2e"]
    assert e["value"] == d["value"] and e["unit"] == d["unit"]
    assert e["h2d_bytes_per_step"] == 0 and e["d2h_bytes_per_step"] == 0
    # tokens/s = batch x 2 tokens per step / mean step time
    B = d["config"]["batch"]
    assert abs(d["value"] - B * 2 / (d["ms_per_step"] * 1e-3)) <= 1e-6 * d["value"]


def test_kernel_bytes_closed_forms():
    """Algorithmic bytes per launch of the 7B-shaped decode classes, written
    out from the weight formats (int8: N K codes + 2 N scales) and the
    activations each launch reads and writes."""
    sys.path.insert(0, ROOT)
    import bench

    t, wq, kvq, B, S, N = bench.CONFIGS["l7b"]
    a = bench.arch_dict(t)
    kb = bench.kernel_bytes(a, wq, kvq, B, S)
    d, f, V = a["hidden"], a["ffn"], a["vocab"]
    qkv = (a["n_heads"] + 2 * a["n_kv_heads"]) * a["head_dim"]
    assert kb["lin_qkv"] == qkv * d + 2 * qkv + 2 * B * (d + qkv)
    assert kb["lin_gu"] == 2 * f * d + 2 * 2 * f + 2 * B * (d + f)
    assert kb["lm_head"] == 2 * V * d + 2 * B * d + 4 * B * V
    # one block's K and V: B x context x Hkv x hd x 2 (K and V) x 2 bytes
    assert kb["attn"] == pytest.approx(B * S * a["n_kv_heads"] * a["head_dim"] * 2 * 2, rel=0.02)


def test_class_roofline_arithmetic():
    """achieved = algorithmic bytes per launch / mean launch time, frac =
    achieved / peak: a class with 2 launches of 100 MB in 0.1 ms in total
    streams 2000 GB/s."""
    sys.path.insert(0, ROOT)
    import bench

    kb = {"lin_gu": 100e6, "attn": 50e6}
    r = bench.class_roofline("lin_gu", kb, {"lin_gu": 0.1, "attn": 0.0}, {"lin_gu": 2, "attn": 0}, 4000.0)
    assert r["launch_ms"] == pytest.approx(0.05)
    assert r["achieved"] == pytest.approx(2000.0)
    assert r["frac"] == pytest.approx(0.5)
    assert r["bytes_per_launch"] == 100e6
    # a class that did not run reports zero rather than dividing by zero
    z = bench.class_roofline("attn", kb, {"lin_gu": 0.1, "attn": 0.0}, {"lin_gu": 2, "attn": 0}, 4000.0)
    assert z["achieved"] == 0.0 and z["frac"] == 0.0


def test_source_code_sha_ignores_comments_only(tmp_path):
    """The recorded ncu traffic stays valid across comment edits of a kernel's
    source and goes stale on any code edit."""
    sys.path.insert(0, ROOT)
    import bench

    base = "// header\n__global__ void k(int* p) {\n  p[0] = 1;  // store\n}\n"
    variants = {
        "same": base,
        "comments": "/* block\n comment */\n// other header\n__global__ void k(int* p) {\n\n  p[0] = 1;\n}\n",
        "code": "// header\n__global__ void k(int* p) {\n  p[0] = 2;  // store\n}\n",
    }
    sha = {}
    for name, text in variants.items():
        f = tmp_path / (name + ".cu")
        f.write_text(text)
        sha[name] = bench.source_code_sha(str(f))
    assert sha["same"] == sha["comments"]
    assert sha["same"] != sha["code"]
    # every table entry names a source that exists
    for (cfg, cls), t in bench.NCU_TRAFFIC.items():
        assert os.path.exists(os.path.join(ROOT, "paper_2501_13111_gb300", "csrc", t["src"])), (cfg, cls)


FAKE_SMI = """#!/bin/bash
# stands in for nvidia-smi: refuses sampling periods below MIN_MS, else prints
# one CSV sample per period (SM MHz counting up from 2000) until killed
for a in "$@"; do last=$a; done
if [ "$last" -lt {min_ms} ]; then echo "Invalid value" >&2; exit 2; fi
sleep 0.2
i=0
while true; do
  echo "0, $((2000 + i)), 2070, 900.00, 0x0, Not Active, Not Active, Not Active, {cap}"
  i=$((i+1)); sleep 0.02
done
"""


@pytest.mark.parametrize("min_ms,cap", [(1, "Active"), (100, "Not Active")])
def test_clock_sampler_samples_inside_the_region(tmp_path, monkeypatch, min_ms, cap):
    """The sampler waits for nvidia-smi's first sample before the timed
    region starts, keeps the samples taken inside it, falls back to a 200 ms
    period when the short one is refused, and reports the power cap."""
    import time

    sys.path.insert(0, ROOT)
    import bench

    smi = tmp_path / "nvidia-smi"
    smi.write_text(FAKE_SMI.format(min_ms=min_ms, cap=cap))
    smi.chmod(0o755)
    monkeypatch.setenv("PATH", f"{tmp_path}:{os.environ['PATH']}")
    with bench.ClockSampler(0) as c:
        time.sleep(0.5)
    s = c.summary()
    assert s["sm_max_mhz"] == 2070.0 and s["samples"] >= 2
    assert all(line.split(",")[1].strip() != "2000" for line in c.lines)  # the pre-region sample is left out
    assert s["reasons"] == (["sw_power_cap"] if cap == "Active" else [])
