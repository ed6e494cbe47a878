"""The traced library (libmpm_trace.so): a merge and a fused compose +
gather leave one (start, waited, end) triple per kernel kind, in order, and
the merge's results equal the ordinary library's.

Runs in a child process, because a process loads one MPM library.
"""

from __future__ import annotations

import json
import os
import subprocess
import sys

import pytest
import torch

pytestmark = pytest.mark.gpu

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))

CHILD = r"""
import json, sys
sys.path.insert(0, sys.argv[1])
import numpy as np, torch
import paper_2604_05718_gb300 as mpm
from paper_2604_05718_gb300 import build
from workloads import make_custom
mpm.library(build.build(trace=True))
b = make_custom([700, 300, 1, 0, 513], 256, "bf16", seed=11)
x = b.tokens.cuda(); off = torch.from_numpy(b.offsets).cuda()
mpm.trace_reset()
x1, off1, m1 = mpm.merge(x, off)
tl1 = mpm.trace_read()
mpm.trace_reset()
x2, off2, m2 = mpm.merge(x1, off1)
up = mpm.compose_gather(x2, off2, m1, off, m2, off1)
tl2 = mpm.trace_read()
t1 = int(off1[-1])
print(json.dumps({"tl1": tl1, "tl2": tl2, "map1": m1[:b.rows].cpu().tolist(), "off1": off1.cpu().tolist(),
                  "x1": x1[:t1].float().cpu().numpy().round(6).tolist()[:50]}))
"""


def test_traced_library_timeline_and_results():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    res = subprocess.run([sys.executable, "-c", CHILD, ROOT], capture_output=True, text=True, timeout=600)
    assert res.returncode == 0, res.stderr[-2000:]
    got = json.loads(res.stdout.strip().splitlines()[-1])
    for tl, kinds in ((got["tl1"], ("prep", "affinity", "mutual_scan", "pair_average")),
                      (got["tl2"], ("prep", "affinity", "mutual_scan", "pair_average", "gather"))):
        assert set(kinds) <= set(tl), tl
        prev_end = 0
        for k in kinds:
            start, waited, end = tl[k]
            assert start <= waited <= end, (k, tl[k])
            assert end - start < 10_000_000, (k, tl[k])    # under 10 ms
            assert waited >= prev_end, (k, tl)               # each kernel waits for the one before it
            prev_end = end
    # Same results as the ordinary library.
    import numpy as np

    import paper_2604_05718_gb300 as mpm
    from paper_2604_05718_gb300 import build
    from workloads import make_custom

    build.build()

    b = make_custom([700, 300, 1, 0, 513], 256, "bf16", seed=11)
    x1, off1, m1 = mpm.merge(b.tokens.cuda(), torch.from_numpy(b.offsets).cuda())
    assert off1.cpu().tolist() == got["off1"]
    assert m1[:b.rows].cpu().tolist() == got["map1"]
    np.testing.assert_array_equal(x1[:int(off1[-1])].float().cpu().numpy().round(6)[:50], np.array(got["x1"]))


def test_bench_timeline_mode():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    res = subprocess.run([sys.executable, os.path.join(ROOT, "bench.py"), "--timeline", "--steps", "2",
                          "--warmup", "1"], capture_output=True, text=True, cwd=ROOT, timeout=900)
    assert res.returncode == 0, res.stderr[-2000:]
    d = json.loads(res.stdout.strip().splitlines()[-1])
    tl = d["timeline"]
    for key in ("prep_1", "affinity_1", "mutual_scan_1", "pair_average_1", "prep_2", "affinity_2",
                "mutual_scan_2", "pair_average_2", "gather"):
        assert tl[key]["us_after_wait"] > 0, key
    assert tl["affinity_1"]["tflops_algorithmic"] > 0 and tl["pair_average_1"]["gbs"] > 0
