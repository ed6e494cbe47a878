"""bench.py's roofline arithmetic on a hand-worked batch (host logic, no GPU).

The figures the JSON line reports (the affinity kernel's algorithmic flop
rate, the bandwidth kernels' byte rates and the whole step against its
combined roofline) are recomputed here by hand for two images of 4 and 3
tokens, D = 8, bf16, two insertions (4, 3 -> 3, 2 -> 2, 2 tokens).
"""

from __future__ import annotations

import importlib.util
import os

import numpy as np
import pytest
import torch

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def bench():
    spec = importlib.util.spec_from_file_location("bench_under_test", os.path.join(ROOT, "bench.py"))
    mod = importlib.util.module_from_spec(spec)
    spec.loader.exec_module(mod)
    return mod


class _Cfg:
    dim, dtype, insertions = 8, "bf16", 2


class _Batch:
    offsets = np.array([0, 4, 7])
    batch, rows = 2, 7


class _Step:
    cfg, batch, two = _Cfg, _Batch, True
    off1_h = np.array([0, 3, 5])
    off2 = torch.tensor([0, 2, 4])


TIMING = {
    "ms": 0.010,  # the step: 10 us
    "kern": {"prep_1_us": 1.0, "pair_average_1_us": 2.0, "prep_2_us": 0.5, "pair_average_2_us": 4.0,
             "compose_gather_us": 2.5, "affinity_1_us": 1.0, "affinity_2_us": 2.0},
    "aff_ms_1": [0.001, 0.001],  # two timed steps: affinity 1 us in stage 1 ...
    "aff_ms_2": [0.002, 0.002],  # ... and 2 us in stage 2
}
PEAKS = {"bf16_tflops": 1000.0, "bf16_tflops_sustained": 800.0, "hbm_gbs": 500.0}


def test_affinity_flops_and_rate(bench):
    m = bench.step_metrics(_Step, TIMING, PEAKS, "measured")
    # N (N - 1) D per image per stage: 4*3*8 + 3*2*8 and 3*2*8 + 2*1*8.
    assert m["alg1"] == 144.0 and m["alg2"] == 64.0
    # Two launches of each stage: (2 * 144 + 2 * 64) flops in 6 us.
    assert m["aff_tflops"] == pytest.approx(416.0 / 6e-6 / 1e12, rel=1e-12)
    assert m["aff_peak_burst"] == 1000.0 and m["aff_peak_sustained"] == 800.0
    # Executed: every image is one tile whose column block holds at most 128
    # tokens, so a narrow 256 x 128 one; K padded to 16.
    assert m["aff_executed_tflops"] == pytest.approx(4 * 2 * 256 * 128 * 2 * 16 / 6e-6 / 1e12, rel=1e-12)


def test_executed_tiles_count_narrow_ones_at_half_width(bench):
    # 862 tokens: R = 4, last block 94 tokens, so its 4 tiles are narrow:
    # 10 - 4 / 2 = 8 full-tile equivalents; 1024 tokens: 10 full tiles;
    # 1100 tokens: R = 5, last block 76: 15 - 5 / 2 = 12.5.
    class Cfg:
        dim, dtype, insertions = 768, "bf16", 1

    class Batch:
        offsets = np.array([0, 862, 1886, 2986])
        batch, rows = 3, 2986

    class Step:
        cfg, batch, two = Cfg, Batch, False
        off1_h = np.array([0, 862, 1886, 2986])
        off2 = None

    t = {"ms": 0.1, "kern": {"prep_1_us": 1.0, "pair_average_1_us": 1.0, "gather_us": 1.0},
         "aff_ms_1": [0.001], "aff_ms_2": []}
    m = bench.step_metrics(Step, t, PEAKS, "measured")
    assert m["aff_executed_tflops"] == pytest.approx((8 + 10 + 12.5) * 256 * 256 * 2 * 768 / 1e-6 / 1e12, rel=1e-12)


def test_bandwidth_kernel_bytes(bench):
    m = bench.step_metrics(_Step, TIMING, PEAKS, "measured")
    hbm = m["hbm"]
    # bytes per row: D * 2 = 16 of tokens; 12 of norm + key (prep) or keys,
    # map and representative list (pair average); gather with two insertions
    # reads both maps and writes the composed one: 12 per grid row.
    expect = {"prep_1": (7 * 16 + 12 * 7, 1.0), "pair_average_1": ((7 + 5) * 16 + 12 * 7, 2.0),
              "prep_2": (5 * 16 + 12 * 5, 0.5), "pair_average_2": ((5 + 4) * 16 + 12 * 5, 4.0),
              "gather": ((4 + 7) * 16 + 12 * 7, 2.5)}
    for name, (nbytes, us) in expect.items():
        assert hbm[f"{name}_gbs"] == pytest.approx(nbytes / (us * 1e-6) / 1e9, rel=1e-12), name
        assert hbm[f"{name}_frac"] == pytest.approx(hbm[f"{name}_gbs"] / 500.0, rel=1e-12), name


def test_whole_step_roofline(bench):
    m = bench.step_metrics(_Step, TIMING, PEAKS, "measured")
    pr = m["pipeline"]
    nbytes = 196 + 276 + 140 + 204 + 260
    assert pr["flops_per_step"] == 208.0 and pr["bytes_per_step"] == nbytes
    tensor_us = 208.0 / 1000e12 * 1e6
    hbm_us = nbytes / 500e9 * 1e6
    assert pr["tensor_us_at_peak"] == pytest.approx(tensor_us, rel=1e-12)
    assert pr["hbm_us_at_peak"] == pytest.approx(hbm_us, rel=1e-12)
    assert pr["measured_us"] == pytest.approx(10.0, rel=1e-12)
    assert pr["frac"] == pytest.approx((tensor_us + hbm_us) / 10.0, rel=1e-12)


def test_workload_summary(bench):
    m = bench.step_metrics(_Step, TIMING, PEAKS, "measured")
    w = bench.workload_summary(_Step, TIMING, m)
    assert w["images_per_s"] == pytest.approx(2 / 10e-6, rel=1e-12)
    assert w["tokens_per_s"] == pytest.approx(7 / 10e-6, rel=1e-12)
    assert w["affinity_frac_of_burst"] == pytest.approx(m["aff_tflops"] / 1000.0, rel=1e-12)
    assert w["pipeline_frac"] == m["pipeline"]["frac"]
    assert w["pair_average_1_frac"] == m["hbm"]["pair_average_1_frac"]
