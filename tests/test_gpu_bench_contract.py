"""bench.py's GPU arm: one JSON line with every field of the contract."""

from __future__ import annotations

import json
import os
import subprocess
import sys

import pytest
import torch

pytestmark = pytest.mark.gpu

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def test_gpu_arm_prints_one_contract_line():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    res = subprocess.run([sys.executable, os.path.join(ROOT, "bench.py"), "--steps", "5", "--warmup", "3",
                          "--no-cpu-baseline", "--no-padded", "--no-chunked", "--no-fp32"],
                         capture_output=True, text=True, cwd=ROOT, timeout=900)
    assert res.returncode == 0, res.stderr[-2000:]
    lines = [ln for ln in res.stdout.splitlines() if ln.strip()]
    assert len(lines) == 1
    d = json.loads(lines[0])
    for key in ("metric", "value", "unit", "n_gpus", "steps", "warmup", "ms_per_step", "higher_is_better",
                "scaling", "vs_baseline", "dtype", "data", "config", "roofline", "e2e", "clocks", "gpu_launches"):
        assert key in d, key
    assert d["n_gpus"] == 1 and d["steps"] == 5 and d["warmup"] == 3 and d["scaling"] == "weak"
    assert d["value"] > 0 and abs(d["value"] * d["ms_per_step"] * 1e-3 - d["config"]["images"]) < 1e-6 * d["value"]
    r = d["roofline"]
    assert r["bound"] == "tensor" and r["unit"] == "TFLOP/s" and 0 < r["frac"] < 1.5
    assert abs(r["frac"] - r["achieved"] / r["peak"]) < 1e-9
    e = d["e2e"]
    assert e["value"] > 0 and e["h2d_bytes_per_step"] > 0 and e["d2h_bytes_per_step"] > 0
    c = d["clocks"]
    assert {"sm_mhz", "sm_max_mhz", "reasons"} <= set(c)
    assert d["gpu_launches"] == 9 * d["steps"]   # four kernels per merge, two merges, one compose + gather
    # Every workload's step, measured in the same run.
    pw = d["per_workload"]
    assert set(pw) == {"vit_t_single", "vit_s", "vit_b", "vit_l", "mixed"}
    for name, w in pw.items():
        assert w["images_per_s"] > 0 and w["tokens_per_s"] > 0, name
        assert 0 < w["affinity_frac_of_burst"] < 1.5 and 0 < w["gather_frac"] < 1.5, name
        assert 0 < w["pair_average_1_frac"] < 1.5 and 0 < w["prep_1_frac"] < 1.5, name
        assert 0 < w["pipeline_frac"] < 1.5, name
    assert abs(pw["vit_b"]["images_per_s"] - d["value"]) < 1e-6 * d["value"]
    # The whole step against its combined tensor + HBM roofline.
    pr = d["pipeline_roofline"]
    assert abs(pr["ideal_us"] - pr["tensor_us_at_peak"] - pr["hbm_us_at_peak"]) < 1e-9 * pr["ideal_us"]
    assert abs(pr["frac"] - pr["ideal_us"] / pr["measured_us"]) < 1e-9 and 0 < pr["frac"] < 1.5
    assert abs(pr["measured_us"] - 1e3 * d["ms_per_step"]) < 1e-6 * pr["measured_us"]
    # The in-step timeline of the traced library, beside the event figures.
    ins = d["in_step"]
    assert ins is not None and ins["affinity_tflops_algorithmic"] > 0
    assert set(ins["kernels_us"]) >= {"prep_1", "affinity_1", "mutual_scan_1", "pair_average_1", "gather"}
