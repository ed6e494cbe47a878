"""Full-size parity on the five synthetic workloads: every image, every stage.

The GPU runs each workload as the benchmark does (whole batch through the C
ABI): merge, the seeded stand-in noise, merge, compose, gather.  Three checks
cover every image:

1. Stage 1: the GPU's merge of the workload against the oracle's
   (``check_image``: bit-exact on decisive rows, valid on near-tie rows).
2. Stage 2, per stage.  The oracle builds its own stage-2 input, its stage-1
   output stored in the I/O dtype plus the seeded noise.  The GPU merges that
   same packed batch in a second call, and every image is checked against the
   oracle's stage 2.  The GPU's compose + gather then run on the oracle's
   stage-1 map and are compared with the oracle's Eq. 3-4 result.  Data flow
   from the oracle to the GPU only; no GPU output ever feeds the oracle.
3. The chained pipeline (stage 2 on the GPU's own stage-1 output).  Where
   stage 1 matched exactly its stage-2 input is bitwise the oracle's, so its
   stage 2, composed map and grid must equal the per-stage result.
   Invariants that hold at any size are checked on every image.

Each workload adds one machine-readable line to the pytest terminal summary.
"""

from __future__ import annotations

import json

import numpy as np
import pytest
import torch

import oracle
from parity import SUMMARY_LINES, ParityStats, check_image, round_to, to_f64
from workloads import CONFIG_ORDER, CONFIGS, DTYPES, apply_noise, make_batch, stage_noise

pytestmark = pytest.mark.gpu

DEV = "cuda"


@pytest.fixture(scope="module")
def mpm():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import paper_2604_05718_gb300 as pkg
    from paper_2604_05718_gb300 import build

    build.build()
    pkg.library()
    return pkg


def gpu_merge(mpm, x: torch.Tensor, offsets: np.ndarray, ws=None) -> dict:
    """nearest neighbours and one merge of a packed batch on the GPU."""
    xd = x.to(DEV)
    off = torch.from_numpy(offsets).to(DEV)
    if ws is None:
        ws = mpm.new_workspace(xd.shape[0], len(offsets) - 1, xd.shape[1], xd.dtype, DEV)
    nn, _ = mpm.nearest_neighbors(xd, off, workspace=ws, with_score=False)
    xo, offo, m = mpm.merge(xd, off, workspace=ws)
    torch.cuda.synchronize()
    assert mpm.device_status(ws) == 0
    offo_h = offo.cpu().numpy()
    return {"x_dev": xo, "off_dev": offo, "map_dev": m, "nn": nn.cpu().numpy(), "map": m.cpu().numpy(),
            "x": to_f64(xo[:offo_h[-1]]), "off": offo_h}


def gpu_pipeline(mpm, batch, cfg) -> dict:
    """The benchmark's step on the GPU, with every intermediate copied out."""
    rows, dim = batch.tokens.shape
    ws = mpm.new_workspace(rows, batch.batch, dim, DTYPES[cfg.dtype], DEV)
    s1 = gpu_merge(mpm, batch.tokens, batch.offsets, ws)
    out = {"s1": s1}
    off0 = torch.from_numpy(batch.offsets).to(DEV)
    if cfg.insertions == 1:
        up = mpm.unmerge_gather(s1["x_dev"], s1["off_dev"], s1["map_dev"], off0)
        out["up"] = to_f64(up[:batch.rows])
        return out
    off1 = s1["off"]
    noise = stage_noise(cfg.seed, np.diff(off1).tolist(), dim).to(DEV)
    x1n = apply_noise(s1["x_dev"][:off1[-1]], noise).contiguous()
    s2 = gpu_merge(mpm, x1n, off1, ws)
    rs = mpm.compose_maps(s1["map_dev"], off0, s2["map_dev"], s1["off_dev"])
    up = mpm.unmerge_gather(s2["x_dev"], s2["off_dev"], rs, off0)
    torch.cuda.synchronize()
    out.update(x1n=to_f64(x1n), s2=s2, rstar=rs.cpu().numpy(), up=to_f64(up[:batch.rows]))
    return out


def check_invariants_all_images(g, batch, cfg) -> None:
    """Properties that hold at any size, on every image of the GPU result."""
    off0, off1 = batch.offsets, g["s1"]["off"]
    for b in range(batch.batch):
        n0 = off0[b + 1] - off0[b]
        n1 = off1[b + 1] - off1[b]
        assert (n0 + 1) // 2 <= n1 <= n0
        m1 = g["s1"]["map"][off0[b]:off0[b + 1]]
        assert n0 == 0 or (m1.min() == 0 and m1.max() == n1 - 1)
        if cfg.insertions == 2:
            off2 = g["s2"]["off"]
            n2 = off2[b + 1] - off2[b]
            assert (n1 + 1) // 2 <= n2 <= n1
            m2 = g["s2"]["map"][off1[b]:off1[b + 1]]
            rs = g["rstar"][off0[b]:off0[b + 1]]
            assert np.array_equal(rs, m2[m1])                          # Eq. 3 on the GPU's maps
            z = g["s2"]["x"][off2[b]:off2[b + 1]]
            assert np.array_equal(g["up"][off0[b]:off0[b + 1]], z[rs])  # Eq. 4 is a pure copy
        else:
            z = g["s1"]["x"][off1[b]:off1[b + 1]]
            assert np.array_equal(g["up"][off0[b]:off0[b + 1]], z[m1])


def _stats_record(st: ParityStats) -> dict:
    return {"images_checked": st.images, "rows": st.rows, "near_tie_rows": st.near_tie_rows,
            "near_tie_deviations": st.nn_deviations, "exact_images": st.images_exact}


@pytest.mark.parametrize("name", CONFIG_ORDER)
def test_workload_parity(mpm, name):
    cfg = CONFIGS[name]
    batch = make_batch(cfg)
    g = gpu_pipeline(mpm, batch, cfg)
    check_invariants_all_images(g, batch, cfg)
    x_all = batch.tokens.double().numpy()
    off0, g_off1 = batch.offsets, g["s1"]["off"]

    # 1. Stage 1 on every image.
    st1, oracle1, exact1 = ParityStats(), [], []
    for b in range(batch.batch):
        a0, a1 = off0[b], off0[b + 1]
        p0, p1 = g_off1[b], g_off1[b + 1]
        st, res, ex = check_image(x_all[a0:a1], g["s1"]["nn"][a0:a1], g["s1"]["map"][a0:a1],
                                  g["s1"]["x"][p0:p1], cfg.dtype, f"{name}[{b}] stage 1")
        st1.add(st)
        oracle1.append(res)
        exact1.append(ex)
    record = {"workload": name, "images": batch.batch, "stage1": _stats_record(st1)}

    if cfg.insertions == 1:
        grid_exact = 0
        for b in range(batch.batch):
            if exact1[b]:
                a0, a1 = off0[b], off0[b + 1]
                want = oracle.gather(round_to(cfg.dtype, oracle1[b].x_out), oracle1[b].r)
                assert np.array_equal(g["up"][a0:a1], want), f"{name}[{b}] reconstructed grid"
                grid_exact += 1
        record["grid_exact_images"] = grid_exact
        _report(record, st1.notes)
        return

    # 2. Stage 2 per stage: the GPU merges the oracle's own stage-2 input.
    counts1 = [r.n_out for r in oracle1]
    off1o = np.concatenate([[0], np.cumsum(counts1)]).astype(np.int64)
    s1o = torch.cat([torch.from_numpy(round_to(cfg.dtype, r.x_out).astype(np.float32)) for r in oracle1])
    x1n_o = apply_noise(s1o.to(DTYPES[cfg.dtype]), stage_noise(cfg.seed, counts1, cfg.dim)).contiguous()
    x1n_o64 = x1n_o.double().numpy()
    g2 = gpu_merge(mpm, x1n_o, off1o)
    st2, oracle2, exact2 = ParityStats(), [], []
    for b in range(batch.batch):
        p0, p1 = off1o[b], off1o[b + 1]
        q0, q1 = g2["off"][b], g2["off"][b + 1]
        st, res, ex = check_image(x1n_o64[p0:p1], g2["nn"][p0:p1], g2["map"][p0:p1], g2["x"][q0:q1],
                                  cfg.dtype, f"{name}[{b}] stage 2")
        st2.add(st)
        oracle2.append(res)
        exact2.append(ex)

    # Compose + gather on the GPU from the oracle's stage-1 map (Eq. 3-4).
    r1_dev = torch.from_numpy(np.concatenate([r.r for r in oracle1]).astype(np.int32)).to(DEV)
    off0_dev, off1o_dev = torch.from_numpy(off0).to(DEV), torch.from_numpy(off1o).to(DEV)
    rs = mpm.compose_maps(r1_dev, off0_dev, g2["map_dev"], off1o_dev)
    up = mpm.unmerge_gather(g2["x_dev"], g2["off_dev"], rs, off0_dev)
    rs_h, up_h = rs.cpu().numpy(), to_f64(up[:batch.rows])
    grid_exact = 0
    for b in range(batch.batch):
        a0, a1 = off0[b], off0[b + 1]
        m2 = g2["map"][off1o[b]:off1o[b + 1]]
        assert np.array_equal(rs_h[a0:a1], m2[oracle1[b].r]), f"{name}[{b}] composed map"
        z = g2["x"][g2["off"][b]:g2["off"][b + 1]]
        assert np.array_equal(up_h[a0:a1], z[rs_h[a0:a1]]), f"{name}[{b}] gather"
        if exact2[b]:
            r_star = oracle.compose(oracle1[b].r, oracle2[b].r)
            assert np.array_equal(rs_h[a0:a1], r_star), f"{name}[{b}] composed map vs oracle"
            want = oracle.gather(round_to(cfg.dtype, oracle2[b].x_out), r_star)
            assert np.array_equal(up_h[a0:a1], want), f"{name}[{b}] reconstructed grid vs oracle"
            grid_exact += 1

    # 3. The chained pipeline equals the per-stage result wherever stage 1 matched.
    chained = 0
    g_off2 = g["s2"]["off"]
    for b in range(batch.batch):
        if not exact1[b]:
            continue
        a0, a1 = off0[b], off0[b + 1]
        gp0, gp1, op0, op1 = g_off1[b], g_off1[b + 1], off1o[b], off1o[b + 1]
        assert np.array_equal(g["x1n"][gp0:gp1], x1n_o64[op0:op1]), f"{name}[{b}] stage-2 input"
        assert np.array_equal(g["s2"]["nn"][gp0:gp1], g2["nn"][op0:op1]), f"{name}[{b}] chained nn"
        assert np.array_equal(g["s2"]["map"][gp0:gp1], g2["map"][op0:op1]), f"{name}[{b}] chained map"
        assert np.array_equal(g["s2"]["x"][g_off2[b]:g_off2[b + 1]], g2["x"][g2["off"][b]:g2["off"][b + 1]])
        assert np.array_equal(g["rstar"][a0:a1], rs_h[a0:a1]), f"{name}[{b}] chained composed map"
        assert np.array_equal(g["up"][a0:a1], up_h[a0:a1]), f"{name}[{b}] chained grid"
        chained += 1
    record.update(stage2=_stats_record(st2), grid_exact_images=grid_exact,
                  chained_images_equal_to_per_stage=chained)
    _report(record, st1.notes + st2.notes)


def _report(record: dict, notes: list) -> None:
    line = "MPM_PARITY " + json.dumps(record, sort_keys=False)
    SUMMARY_LINES.append(line)
    print("\n" + line)
    for note in notes:
        print("  " + note)
