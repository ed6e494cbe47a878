#!/usr/bin/env python
"""Throughput of the MPM hot path on one GB300 per rank.

A step is one pass of the whole path over one batch of synthetic tokens:
merge (Algorithm 1) -> merge -> compose maps (Eq. 3) -> gather (Eq. 4).
Between the two merges a seeded N(0, 0.05^2) perturbation stands in for the
encoder blocks; it is not part of MPM and is not timed.

  python bench.py [--gpus N] [--steps K] [--warmup W] [--workload vit_b]
  python bench.py --impl reference ...   # the fp64 CPU oracle on host cores

Timing: CUDA events on the launch stream bracket the two timed segments of
every step (merge 1; merge 2 + compose + gather).  A second timed loop adds
events around every kernel for the per-kernel breakdown and the roofline
(those events serialise the kernels, so the step time comes from the first); L2 is flushed before every
step by writing and then reading a 256 MiB buffer; W untimed warm-up steps; barrier + synchronize on
both sides; the max over ranks is reported.  Each rank processes its own
batch (images are independent: replicas, weak scaling, no collective on the
data path).  One JSON line is printed by rank 0.
"""

from __future__ import annotations

import argparse
import hashlib
import json
import os
import platform
import statistics
import sys
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

METRIC = "MPM images/sec (merge+compose+unmerge); % bf16 tensor peak, % HBM BW"
UNIT = "images/s"
DEFAULT_WORKLOAD = "vit_b"
PEAKS_FILE = os.path.join(ROOT, "MEASURED_PEAKS.json")
# Fallback denominators when the measured file is absent.
FALLBACK_PEAKS = {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0}
L2_FLUSH_BYTES = 256 << 20
KERNELS_PER_MERGE = 4
TRAFFIC_FILE = os.path.join(ROOT, "profiles", "affinity_pair_traffic.txt")
# The sources the affinity kernel is compiled from; the traffic record holds
# a hash of their concatenation.
AFFINITY_SOURCES = [os.path.join(ROOT, "paper_2604_05718_gb300", "csrc", f)
                    for f in ("affinity_pair.cu", "affinity_epilogue.cuh", "ptx.cuh", "common.cuh")]


def parse_args():
    p = argparse.ArgumentParser(description=__doc__, formatter_class=argparse.RawDescriptionHelpFormatter)
    p.add_argument("--gpus", type=int, default=1)
    p.add_argument("--steps", type=int, default=200)
    p.add_argument("--warmup", type=int, default=10)
    p.add_argument("--impl", choices=["mpm", "reference"], default="mpm")
    p.add_argument("--workload", default=DEFAULT_WORKLOAD)
    p.add_argument("--no-cpu-baseline", action="store_true")
    p.add_argument("--cpu-seconds", type=float, default=12.0, help="target wall time of the oracle sample")
    p.add_argument("--no-e2e", action="store_true")
    p.add_argument("--no-chunked", action="store_true", help="skip the chunked-similarity measurement")
    p.add_argument("--no-padded", action="store_true", help="skip the padded-batch measurement")
    p.add_argument("--no-fp32", action="store_true", help="skip the fp32 nearest-neighbour measurement")
    p.add_argument("--no-per-workload", action="store_true",
                   help="skip the step on the other four workloads (per_workload in the JSON line)")
    p.add_argument("--no-timeline", action="store_true",
                   help="skip the in-step device timeline (traced library, child process) of the default run")
    p.add_argument("--timeline", action="store_true",
                   help="instead of the benchmark, print each kernel's in-step duration from the device "
                        "timeline of the traced library (libmpm_trace.so); one GPU")
    return p.parse_args()


def dist_env():
    rank = int(os.environ.get("RANK", "0"))
    world = int(os.environ.get("WORLD_SIZE", "1"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return rank, world, local


def load_peaks():
    try:
        with open(PEAKS_FILE) as f:
            pk = json.load(f)
        return pk, "measured"
    except (OSError, ValueError):
        return dict(FALLBACK_PEAKS), "fallback"


def workload_desc(cfg, batch, world=1):
    sizes = np.diff(batch.offsets)
    return {
        "workload": f"{cfg.name}: {cfg.description}",
        "images": int(world * cfg.batch),
        "images_this_rank": int(batch.batch),
        "tokens_this_rank": int(batch.rows),
        "tokens_per_image": int(sizes[0]) if len(set(sizes.tolist())) == 1 else "mixed",
        "dim": int(cfg.dim),
        "insertions": int(cfg.insertions),
        "seed": int(cfg.seed),
        "l2": "flushed before every step: 256 MiB written, then read back (clean lines)",
        "untimed": "the seeded N(0,0.05^2) stand-in for the encoder blocks between the two merges",
        "parallelism": "image shards: each rank merges one contiguous range of the world*B images, "
                       "balanced on sum(N_b^2) (shard.partition_images); no data-path collective",
    }


# ---------------------------------------------------------------------------
# The fp64 oracle on the host cores (cpu_baseline leg and --impl reference)
# ---------------------------------------------------------------------------
def oracle_image_pipeline(cfg, x_img, b):
    """merge -> noise -> merge -> compose -> gather for one image (oracle)."""
    import torch

    import oracle
    from workloads import DTYPES, apply_noise, stage_noise

    def stored(v):
        return oracle.round_bf16(v) if cfg.dtype == "bf16" else oracle.round_f32(v).astype(np.float64)

    m1 = oracle.merge_image(x_img)
    if cfg.insertions == 1:
        return oracle.gather(stored(m1.x_out), m1.r)
    s1 = torch.from_numpy(stored(m1.x_out).astype(np.float32)).to(DTYPES[cfg.dtype])
    noise = stage_noise(cfg.seed, [m1.n_out], cfg.dim, images=[b])
    s1n = apply_noise(s1, noise).double().numpy()
    m2 = oracle.merge_image(s1n)
    r_star = oracle.compose(m1.r, m2.r)
    return oracle.gather(stored(m2.x_out), r_star)


def oracle_sample(cfg, batch, seconds):
    """Times the oracle over the workload's images, in order and wrapping
    around, until about `seconds` of wall time have passed."""
    x = batch.tokens.double().numpy()
    t0 = time.perf_counter()
    done = 0
    while True:
        b = done % cfg.batch
        oracle_image_pipeline(cfg, x[batch.offsets[b]:batch.offsets[b + 1]], b)
        done += 1
        if time.perf_counter() - t0 > seconds:
            break
    dt = time.perf_counter() - t0
    return done, dt


def host_cores():
    try:
        return len(os.sched_getaffinity(0))
    except AttributeError:
        return os.cpu_count() or 1


def cpu_baseline_obj(images, seconds, cfg):
    return {
        "value": images / seconds,
        "unit": UNIT,
        "cores": host_cores(),
        "kind": "oracle",
        "sample": (f"{images} image pipelines over the {cfg.batch} images of {cfg.name} "
                   f"({images / cfg.batch:.2f} passes), full pipeline per image "
                   f"(merge, stand-in noise, merge, compose, gather) in fp64 numpy, {seconds:.1f} s wall; "
                   f"BLAS threads default, {platform.machine()} host"),
    }


def run_reference(args):
    rank, world, _ = dist_env()
    if rank != 0:
        return 0
    from workloads import CONFIGS, make_batch

    cfg = CONFIGS[args.workload]
    batch = make_batch(cfg)
    x = batch.tokens.double().numpy()
    for s in range(args.warmup):
        b = s % cfg.batch
        oracle_image_pipeline(cfg, x[batch.offsets[b]:batch.offsets[b + 1]], b)
    t0 = time.perf_counter()
    for s in range(args.steps):
        b = (args.warmup + s) % cfg.batch
        oracle_image_pipeline(cfg, x[batch.offsets[b]:batch.offsets[b + 1]], b)
    dt = time.perf_counter() - t0
    value = args.steps / dt
    line = {
        "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": args.gpus, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": 1e3 * dt / args.steps, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
        "config": dict(workload_desc(cfg, batch), step="one image of the workload per step"),
        "impl": "reference",
        "cpu_baseline": dict(cpu_baseline_obj(args.steps, dt, cfg)),
        "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)
    return 0


# ---------------------------------------------------------------------------
# Clock sampling during the timed region
# ---------------------------------------------------------------------------
class ClockSampler:
    """SM clock and throttle reasons sampled during the timed region.

    Reads NVML through ctypes (read-only queries: current and maximum SM
    clock, clock event reasons) every millisecond from a thread, so that even
    a timed region of a few milliseconds gets samples.  Falls back to
    nothing (clocks null) when NVML is not available.
    """

    REASONS = {0x4: "sw_power_cap", 0x8: "hw_slowdown", 0x20: "sw_thermal_slowdown",
               0x40: "hw_thermal_slowdown", 0x80: "hw_power_brake_slowdown"}

    def __init__(self, torch_device):
        import ctypes
        import threading

        self.ok = False
        self.samples = []
        self.max_mhz = None
        self._stop = threading.Event()
        self._thread = None
        try:
            nvml = ctypes.CDLL("libnvidia-ml.so.1")
            if nvml.nvmlInit_v2() != 0:
                return
            handle = ctypes.c_void_p()
            bus = self._bus_id(torch_device)
            if bus is None or nvml.nvmlDeviceGetHandleByPciBusId_v2(bus.encode(), ctypes.byref(handle)) != 0:
                if nvml.nvmlDeviceGetHandleByIndex_v2(torch_device.index or 0, ctypes.byref(handle)) != 0:
                    return
            mx = ctypes.c_uint(0)
            if nvml.nvmlDeviceGetMaxClockInfo(handle, 1, ctypes.byref(mx)) == 0:  # 1 = SM clock
                self.max_mhz = float(mx.value)
            self.reasons_fn = getattr(nvml, "nvmlDeviceGetCurrentClocksEventReasons", None) or \
                getattr(nvml, "nvmlDeviceGetCurrentClocksThrottleReasons")
            self.nvml, self.handle, self.ok = nvml, handle, True
        except (OSError, AttributeError):
            self.ok = False

    @staticmethod
    def _bus_id(dev):
        import torch

        props = torch.cuda.get_device_properties(dev)
        try:
            return f"{props.pci_domain_id:08X}:{props.pci_bus_id:02X}:{props.pci_device_id:02X}.0"
        except AttributeError:
            return None

    def _run(self):
        import ctypes

        clk = ctypes.c_uint(0)
        rsn = ctypes.c_ulonglong(0)
        while not self._stop.is_set():
            if self.nvml.nvmlDeviceGetClockInfo(self.handle, 1, ctypes.byref(clk)) == 0:
                bits = rsn.value if self.reasons_fn(self.handle, ctypes.byref(rsn)) == 0 else 0
                self.samples.append((float(clk.value), int(bits)))
            time.sleep(0.001)

    def start(self):
        if not self.ok:
            return
        import threading

        self._thread = threading.Thread(target=self._run, daemon=True)
        self._thread.start()
        t0 = time.perf_counter()
        while not self.samples and time.perf_counter() - t0 < 1.0:
            time.sleep(0.001)

    def stop(self):
        if not self.ok or self._thread is None:
            return None
        self._stop.set()
        self._thread.join(timeout=5)
        if not self.samples:
            return None
        reasons = set()
        for _, bits in self.samples:
            for bit, name in self.REASONS.items():
                if bits & bit:
                    reasons.add(name)
        sm = [c for c, _ in self.samples]
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": self.max_mhz, "reasons": sorted(reasons),
                "samples": len(sm), "source": "NVML, 1 ms period, during the timed steps"}


def kernel_sources_sha(files) -> str:
    """First 16 hex digits of the SHA-256 of the files' concatenated bytes."""
    h = hashlib.sha256()
    for name in files:
        with open(name, "rb") as f:
            h.update(f.read())
    return h.hexdigest()[:16]


def traffic_for(kernel_files, rows_per_launch: float):
    """DRAM bytes per launch from the committed ncu record, if the kernel is unchanged.

    The record holds one captured launch's dram read + write bytes and its
    rows; the kernel reads its input once, so the bytes scale with the rows.
    """
    try:
        with open(TRAFFIC_FILE) as f:
            fields = dict(line.strip().split("=", 1) for line in f if "=" in line and not line.startswith("#"))
        if fields.get("source_sha256_16") == kernel_sources_sha(kernel_files):
            per_row = (float(fields["dram_read_bytes"]) + float(fields["dram_write_bytes"])) / \
                float(fields["rows_captured"])
            return per_row * rows_per_launch
    except (OSError, ValueError, KeyError):
        pass
    return None


# ---------------------------------------------------------------------------
# The GPU path
# ---------------------------------------------------------------------------
# Nominal dense tf32 / bf16 tensor throughput (1.1 / 2.25 PFLOP/s per GB300):
# the fp32 path's peak is the measured bf16 peak times this ratio.
TF32_PER_BF16 = 1.1 / 2.25


def new_events(stream, n):
    """n timing events, recorded once so that their CUDA handles exist."""
    import torch

    evs = [torch.cuda.Event(enable_timing=True) for _ in range(n)]
    for e in evs:
        e.record(stream)
    return evs


class StepEvents:
    """The CUDA events of one step."""

    def __init__(self, stream):
        self.seg = new_events(stream, 4)   # [merge1 start, merge1 end, rest start, rest end]
        self.k1 = new_events(stream, 8)    # merge 1 kernels
        self.k2 = new_events(stream, 8)    # merge 2 kernels
        self.cg = new_events(stream, 2)    # around the (composed) gather


class Step:
    """Device buffers of one packed batch and the launches of one step.

    merge (Algorithm 1) -> the untimed stand-in noise -> merge -> compose and
    gather in one pass (Eq. 3 + Eq. 4); one insertion: merge -> gather.
    """

    def __init__(self, mpm, cfg, batch, images, dev, stream, flush, flush_sum):
        import torch

        from workloads import stage_noise

        self.mpm, self.cfg, self.batch, self.stream = mpm, cfg, batch, stream
        self.flush, self.flush_sum = flush, flush_sum
        rows, dim, nimg = batch.rows, cfg.dim, batch.batch
        self.x0 = batch.tokens.to(dev)
        self.off0 = torch.from_numpy(batch.offsets).to(dev)
        self.ws = mpm.new_workspace(rows, nimg, dim, self.x0.dtype, dev)
        self.x1 = torch.empty_like(self.x0)
        self.off1 = torch.empty(nimg + 1, dtype=torch.int64, device=dev)
        self.m1 = torch.empty(rows, dtype=torch.int32, device=dev)
        self.x1n = torch.zeros_like(self.x0)
        self.x2 = torch.empty_like(self.x0)
        self.off2 = torch.empty_like(self.off1)
        self.m2 = torch.empty_like(self.m1)
        self.rstar = torch.empty_like(self.m1)
        self.up = torch.empty_like(self.x0)
        self.two = cfg.insertions == 2
        # One untimed pass fixes the stage-1 counts, hence the stand-in noise.
        mpm.merge(self.x0, self.off0, workspace=self.ws, out_tokens=self.x1, out_offsets=self.off1,
                  out_map=self.m1)
        self.off1_h = self.off1.cpu().numpy()
        self.t1 = int(self.off1_h[-1])
        self.noise = (stage_noise(cfg.seed, np.diff(self.off1_h).tolist(), dim, images=images).to(dev)
                      if self.two else None)

    def launches(self) -> int:
        """Kernels of the library launched by one step."""
        return 2 * KERNELS_PER_MERGE + 1 if self.two else KERNELS_PER_MERGE + 1

    def run(self, ev: StepEvents, host_in=None, host_out=None, per_kernel=False):
        """One step; per_kernel adds CUDA events between the kernels (which
        serialises them, so the step time is taken without them)."""
        from workloads import apply_noise

        mpm, s = self.mpm, self.stream
        # Evict the L2: write 256 MiB, then read it back so that the lines left
        # behind are clean (no write-back lands on the first timed kernel).
        self.flush.fill_(1)
        self.flush_sum.copy_(self.flush.view(self.flush_sum.dtype).sum())
        ev.seg[0].record(s)
        if host_in is not None:
            self.x0.copy_(host_in[0], non_blocking=True)
            self.off0.copy_(host_in[1], non_blocking=True)
        mpm.merge(self.x0, self.off0, workspace=self.ws, out_tokens=self.x1, out_offsets=self.off1,
                  out_map=self.m1, stage_events=ev.k1 if per_kernel else None)
        ev.seg[1].record(s)
        if self.two:
            self.x1n[:self.t1] = apply_noise(self.x1[:self.t1], self.noise)
        ev.seg[2].record(s)
        if self.two:
            mpm.merge(self.x1n, self.off1, workspace=self.ws, out_tokens=self.x2, out_offsets=self.off2,
                      out_map=self.m2, stage_events=ev.k2 if per_kernel else None)
            if per_kernel:
                ev.cg[0].record(s)
            # Eq. 3 and Eq. 4 in one pass; rstar receives the composed map.
            mpm.compose_gather(self.x2, self.off2, self.m1, self.off0, self.m2, self.off1, out=self.up,
                               out_map=self.rstar)
        else:
            if per_kernel:
                ev.cg[0].record(s)
            mpm.unmerge_gather(self.x1, self.off1, self.m1, self.off0, out=self.up)
        if per_kernel:
            ev.cg[1].record(s)
        if host_out is not None:
            host_out.copy_(self.up, non_blocking=True)
        ev.seg[3].record(s)


def time_step(p: Step, steps: int, warmup: int, barrier, max_over_ranks, clocks=None) -> dict:
    """W warm-up steps, then K timed steps without and K with per-kernel events.

    Returns the mean step time (max over ranks), the per-kernel means and
    the affinity kernel's per-launch durations.
    """
    warm = StepEvents(p.stream)
    for _ in range(warmup):
        p.run(warm)
    assert p.mpm.device_status(p.ws) == 0, "device status reported an error during warm-up"
    events = [StepEvents(p.stream) for _ in range(steps)]
    barrier()
    if clocks is not None:
        clocks.start()
    wall0 = time.perf_counter()
    for ev in events:
        p.run(ev)
    barrier()
    wall = time.perf_counter() - wall0
    clk = clocks.stop() if clocks is not None else None
    seg_ms = [ev.seg[0].elapsed_time(ev.seg[1]) + ev.seg[2].elapsed_time(ev.seg[3]) for ev in events]
    ms = max_over_ranks(statistics.mean(seg_ms))
    assert p.mpm.device_status(p.ws) == 0, "device status reported an error in the timed loop"

    # Second timed loop, same steps with CUDA events around every kernel: the
    # per-kernel durations for the roofline and the breakdown.
    kevents = [StepEvents(p.stream) for _ in range(steps)]
    barrier()
    for ev in kevents:
        p.run(ev, per_kernel=True)
    barrier()
    ms_k = max_over_ranks(statistics.mean(
        [ev.seg[0].elapsed_time(ev.seg[1]) + ev.seg[2].elapsed_time(ev.seg[3]) for ev in kevents]))

    def kernel_ms(key, k):
        return [getattr(ev, key)[2 * k].elapsed_time(getattr(ev, key)[2 * k + 1]) for ev in kevents]

    kern = {}
    for k, nm in enumerate(["prep", "affinity", "mutual_scan", "pair_average"]):
        kern[f"{nm}_1_us"] = 1e3 * statistics.mean(kernel_ms("k1", k))
        if p.two:
            kern[f"{nm}_2_us"] = 1e3 * statistics.mean(kernel_ms("k2", k))
    cg = [ev.cg[0].elapsed_time(ev.cg[1]) for ev in kevents]
    kern["compose_gather_us" if p.two else "gather_us"] = 1e3 * statistics.mean(cg)
    return {"ms": ms, "wall": wall, "clocks": clk, "ms_with_kernel_events": ms_k, "kern": kern,
            "aff_ms_1": kernel_ms("k1", 1), "aff_ms_2": kernel_ms("k2", 1) if p.two else []}


def step_metrics(p: Step, t: dict, peaks: dict, peak_kind: str) -> dict:
    """Roofline figures of a timed step: the affinity kernel's algorithmic
    flop rate and the bandwidth kernels' algorithmic byte rates."""
    cfg, dim, kern = p.cfg, p.cfg.dim, t["kern"]
    esize = 2 if cfg.dtype == "bf16" else 4
    n0 = np.diff(p.batch.offsets).astype(np.float64)
    n1 = np.diff(p.off1_h).astype(np.float64)
    n2 = np.diff(p.off2.cpu().numpy()).astype(np.float64) if p.two else n1
    # Algorithmic work of the affinity step: S is symmetric with a masked
    # diagonal, so the minimum is the N(N-1)/2 off-diagonal dot products of
    # D multiply-adds each, N(N-1)D flops per image per stage.
    alg1 = float(np.sum(n0 * (n0 - 1.0) * dim))
    alg2 = float(np.sum(n1 * (n1 - 1.0) * dim)) if p.two else 0.0
    aff_ms = t["aff_ms_1"] + t["aff_ms_2"]
    aff_flops = [alg1] * len(t["aff_ms_1"]) + [alg2] * len(t["aff_ms_2"])
    achieved = sum(aff_flops) / (sum(aff_ms) * 1e-3) / 1e12
    ratio = 1.0 if cfg.dtype == "bf16" else TF32_PER_BF16
    burst = ratio * peaks.get("bf16_tflops", FALLBACK_PEAKS["bf16_tflops"])
    sustained = ratio * peaks.get("bf16_tflops_sustained", FALLBACK_PEAKS["bf16_tflops_sustained"])
    # What the tensor pipe executes (bf16): the 256 x 256 tiles on or above
    # each image's diagonal, over K padded to 16 (the MMA's K).  The R tiles
    # of an image's last column block are narrow (256 x 128) when that block
    # holds at most 128 of its tokens.
    kpad = -(-dim // 16) * 16

    def exec_flops(ns):
        n = ns.astype(np.int64)
        r = -(-n // 256)
        narrow = (n > 0) & (n - 256 * (r - 1) <= 128)
        tiles = r * (r + 1) / 2.0 - np.where(narrow, r / 2.0, 0.0)
        return float(np.sum(tiles)) * 256 * 256 * 2 * kpad

    exe = [exec_flops(n0)] * len(t["aff_ms_1"]) + [exec_flops(n1)] * len(t["aff_ms_2"])
    executed = sum(exe) / (sum(aff_ms) * 1e-3) / 1e12 if cfg.dtype == "bf16" else None
    hbm = peaks.get("hbm_gbs", FALLBACK_PEAKS["hbm_gbs"])

    def gbs(nbytes, us):
        return nbytes / (us * 1e-6) / 1e9

    # Algorithmic bytes of the bandwidth kernels.  prep reads the tokens and
    # writes a norm and a key reset per row; pair average reads every input
    # row once, writes the merged rows and moves 12 bytes of keys, map and
    # representative list per input row (the mutual scan's traffic, counted
    # here); gather reads each merged row it needs and writes the grid, and
    # with two insertions also reads both maps and writes the composed one.
    nbytes = {
        "prep_1": n0.sum() * dim * esize + 12 * n0.sum(),
        "pair_average_1": (n0.sum() + n1.sum()) * dim * esize + 12 * n0.sum(),
    }
    if p.two:
        nbytes["prep_2"] = n1.sum() * dim * esize + 12 * n1.sum()
        nbytes["pair_average_2"] = (n1.sum() + n2.sum()) * dim * esize + 12 * n1.sum()
    nbytes["gather"] = (n2.sum() + n0.sum()) * dim * esize + (12 if p.two else 4) * n0.sum()
    kern_us = dict((k, kern[f"{k}_us"]) for k in nbytes if k != "gather")
    kern_us["gather"] = kern["compose_gather_us" if p.two else "gather_us"]
    bw = {f"{k}_gbs": gbs(v, kern_us[k]) for k, v in nbytes.items()}
    for k in list(bw):
        bw[k.replace("_gbs", "_frac")] = bw[k] / hbm
    # The whole step against its roofline: the time the affinity flops need
    # at the tensor peak plus the time the bandwidth kernels' bytes need at
    # the copy bandwidth, over the measured step time.
    flops_step = alg1 + alg2
    bytes_step = float(sum(nbytes.values()))
    tensor_us = flops_step / (burst * 1e12) * 1e6
    hbm_us = bytes_step / (hbm * 1e9) * 1e6
    pipeline = {"flops_per_step": flops_step, "bytes_per_step": bytes_step,
                "tensor_us_at_peak": tensor_us, "hbm_us_at_peak": hbm_us,
                "ideal_us": tensor_us + hbm_us, "measured_us": 1e3 * t["ms"],
                "frac": (tensor_us + hbm_us) / (1e3 * t["ms"]),
                "definition": "(algorithmic affinity flops / bf16 burst peak + algorithmic bytes of prep, "
                              "pair average and gather / measured copy bandwidth) / step time"}
    return {"n0": n0, "n1": n1, "n2": n2, "alg1": alg1, "alg2": alg2,
            "aff_launches": len(aff_ms), "aff_flops_per_launch": sum(aff_flops) / len(aff_ms),
            "aff_tflops": achieved, "aff_peak_burst": burst, "aff_peak_sustained": sustained,
            "aff_executed_tflops": executed, "hbm": bw, "hbm_peak": hbm, "pipeline": pipeline,
            "rows_per_aff_launch": (n0.sum() + (n1.sum() if p.two else 0.0)) / (2.0 if p.two else 1.0)}


def workload_summary(p: Step, t: dict, m: dict) -> dict:
    """The per-workload record of the JSON line."""
    out = {
        "images": p.batch.batch, "tokens": p.batch.rows, "dim": p.cfg.dim, "dtype": p.cfg.dtype,
        "insertions": p.cfg.insertions, "ms_per_step": t["ms"],
        "images_per_s": p.batch.batch / (t["ms"] * 1e-3), "tokens_per_s": p.batch.rows / (t["ms"] * 1e-3),
        "affinity_tflops_algorithmic": m["aff_tflops"],
        "affinity_frac_of_burst": m["aff_tflops"] / m["aff_peak_burst"],
        "affinity_frac_of_sustained": m["aff_tflops"] / m["aff_peak_sustained"],
        "affinity_peak": ("bf16 dense" if p.cfg.dtype == "bf16" else
                          "tf32 dense = bf16 x 1.1/2.25 (nominal ratio); three tf32 products per term"),
        "affinity_us": {k: v for k, v in t["kern"].items() if k.startswith("affinity")},
        "pipeline_frac": m["pipeline"]["frac"],
    }
    out.update({k: v for k, v in m["hbm"].items() if k.endswith("_frac")})
    return out


def run_mpm(args):
    import torch
    import torch.distributed as dist

    import paper_2604_05718_gb300 as mpm
    from paper_2604_05718_gb300 import build
    from paper_2604_05718_gb300.shard import partition_images
    from workloads import CONFIG_ORDER, CONFIGS, WorkloadConfig, apply_noise, image_shape, make_batch

    rank, world, local = dist_env()
    if not torch.cuda.is_available():
        raise RuntimeError("bench.py needs a CUDA device")
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    if world > 1:
        dist.init_process_group("nccl", device_id=dev)
    build.build()
    mpm.library()

    cfg = CONFIGS[args.workload]
    # The global batch holds world x B images of the workload.  Rank r merges
    # one contiguous range of them, balanced on sum(N_b^2) (the affinity
    # cost); images are independent, so no data crosses ranks.
    global_images = world * cfg.batch
    sizes = [image_shape(cfg, b)[0] ** 2 for b in range(global_images)]
    lo, hi = partition_images(sizes, world)[rank]
    if hi <= lo:
        raise RuntimeError(f"rank {rank} received no images of the {global_images}-image batch")
    images = list(range(lo, hi))
    batch = make_batch(cfg, images=images)
    rows, dim, nimg = batch.rows, cfg.dim, batch.batch
    esize = 2 if cfg.dtype == "bf16" else 4
    stream = torch.cuda.current_stream(dev)

    # CPU baseline first (pure numpy, rank 0, one GPU only), before GPU work.
    cpu_base = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        n_img, secs = oracle_sample(cfg, batch, args.cpu_seconds)
        cpu_base = cpu_baseline_obj(n_img, secs, cfg)

    flush = torch.empty(L2_FLUSH_BYTES, dtype=torch.uint8, device=dev)
    flush_sum = torch.zeros((), dtype=torch.int64, device=dev)
    p = Step(mpm, cfg, batch, images, dev, stream, flush, flush_sum)
    x0, off0, ws, x1, off1, m1 = p.x0, p.off0, p.ws, p.x1, p.off1, p.m1
    x1n, x2, off2, m2, rstar, up = p.x1n, p.x2, p.off2, p.m2, p.rstar, p.up
    t1, two, noise = p.t1, p.two, p.noise

    def barrier():
        torch.cuda.synchronize(dev)
        if world > 1:
            dist.barrier()
        torch.cuda.synchronize(dev)

    def max_over_ranks(v: float) -> float:
        if world == 1:
            return v
        t = torch.tensor([v], dtype=torch.float64, device=dev)
        dist.all_reduce(t, op=dist.ReduceOp.MAX)
        return float(t.item())

    # ---------------- device-resident timed loop ----------------
    t = time_step(p, args.steps, args.warmup, barrier, max_over_ranks, ClockSampler(dev))
    ms, wall, clk, kern = t["ms"], t["wall"], t["clocks"], t["kern"]
    ms_with_kernel_events = t["ms_with_kernel_events"]
    peaks, peak_kind = load_peaks()
    m = step_metrics(p, t, peaks, peak_kind)
    n0, n1, n2 = m["n0"], m["n1"], m["n2"]
    roofline = {
        "kernel": "affinity_pair_kernel (fused cosine affinity + arg max, TMA + tcgen05.mma.cta_group::2)",
        "bound": "tensor", "achieved": m["aff_tflops"], "peak": m["aff_peak_burst"], "unit": "TFLOP/s",
        "frac": m["aff_tflops"] / m["aff_peak_burst"],
        "peak_kind": (f"{peak_kind} bf16 burst: the timed region is {args.steps} steps of well under a "
                      "millisecond each, not a seconds-long loop"),
        "peak_sustained": m["aff_peak_sustained"],
        "frac_of_sustained": m["aff_tflops"] / m["aff_peak_sustained"],
        "flops_per_launch": m["aff_flops_per_launch"],
        "flops_definition": "algorithmic: N_b (N_b - 1) D per image per stage (off-diagonal half of S = X X^T)",
        "executed_tflops": m["aff_executed_tflops"],
        "executed_frac": (m["aff_executed_tflops"] / m["aff_peak_burst"]
                          if m["aff_executed_tflops"] is not None else None),
        "executed_definition": ("MMA work issued: 256x256 tiles on or above the diagonal (256x128 where the "
                                "column block holds at most 128 tokens) x K padded to 16"),
        "traffic": traffic_for(AFFINITY_SOURCES, m["rows_per_aff_launch"]),
    }
    hbm_kernels = dict(m["hbm"], peak_gbs=m["hbm_peak"], peak_kind=f"{peak_kind} copy bandwidth")

    # ---------------- every workload, the same step (one GPU) ----------------
    per_workload = None
    if world == 1 and not args.no_per_workload:
        per_workload = {}
        pw_steps, pw_warm = min(args.steps, 50), max(3, min(args.warmup, 5))
        for name in CONFIG_ORDER:
            if name == args.workload:
                per_workload[name] = dict(workload_summary(p, t, m), steps=args.steps)
                continue
            wcfg = CONFIGS[name]
            wb = make_batch(wcfg)
            wp = Step(mpm, wcfg, wb, list(range(wcfg.batch)), dev, stream, flush, flush_sum)
            wt = time_step(wp, pw_steps, pw_warm, barrier, max_over_ranks)
            per_workload[name] = dict(workload_summary(wp, wt, step_metrics(wp, wt, peaks, peak_kind)),
                                      steps=pw_steps)
            del wp, wb

    # ---------------- padded batch of the stage-1 output (next-step consumer layout) ----------------
    # The merged sequences padded to the longest one, with a key mask, as the
    # paper batches them for dense attention; and back to the packed layout.
    padded = None
    n1_max = int(n1.max())
    pad_out = torch.empty(nimg, n1_max, dim, dtype=x1.dtype, device=dev) if not args.no_padded else None
    pad_mask = torch.empty(nimg, n1_max, dtype=torch.uint8, device=dev)
    pad_stats = torch.empty(3, dtype=torch.int64, device=dev)
    unpadded = torch.empty_like(x1) if not args.no_padded else None
    pad_us, unpad_us = [], []
    for it in range(0 if args.no_padded else max(3, args.warmup) + 20):
        flush.fill_(1)
        flush_sum.copy_(flush.view(torch.int64).sum())
        e = new_events(stream, 3)
        e[0].record(stream)
        mpm.pad_batch(x1, off1, n1_max, out=pad_out, mask=pad_mask, stats=pad_stats)
        e[1].record(stream)
        mpm.unpad_batch(pad_out, off1, out=unpadded)
        e[2].record(stream)
        if it >= max(3, args.warmup):
            torch.cuda.synchronize(dev)
            pad_us.append(1e3 * e[0].elapsed_time(e[1]))
            unpad_us.append(1e3 * e[1].elapsed_time(e[2]))
    hbm_bw = peaks.get("hbm_gbs", FALLBACK_PEAKS["hbm_gbs"])
    pad_bytes = float(n1.sum() * dim * esize + nimg * n1_max * (dim * esize + 1))
    unpad_bytes = float(2 * n1.sum() * dim * esize)
    if not args.no_padded:
        assert torch.equal(unpadded[:t1], x1[:t1]), "unpad(pad(x)) differs from x"
        padded = {
            "L": n1_max, "rows": int(n1.sum()), "padding_frac": 1.0 - float(n1.sum()) / (nimg * n1_max),
            "pad_us": statistics.median(pad_us), "unpad_us": statistics.median(unpad_us),
            "pad_gbs": pad_bytes / (statistics.median(pad_us) * 1e-6) / 1e9,
            "unpad_gbs": unpad_bytes / (statistics.median(unpad_us) * 1e-6) / 1e9,
        }
        padded["pad_frac"] = padded["pad_gbs"] / hbm_bw
        padded["unpad_frac"] = padded["unpad_gbs"] / hbm_bw

    # ---------------- chunked similarity on the mixed-resolution workload ----------------
    # One merge of the mixed workload (1024-4096 tokens per image) with the
    # full similarity and with chunks of 1024 tokens (mpm_merge_chunked).
    chunked = None
    if rank == 0 and not args.no_chunked:
        mcfg = CONFIGS["mixed"]
        mb = make_batch(mcfg)
        mx = mb.tokens.to(dev)
        moff = torch.from_numpy(mb.offsets).to(dev)
        mws = mpm.new_workspace(mb.rows, mcfg.batch, mcfg.dim, mx.dtype, dev)
        mout = torch.empty_like(mx)
        moo = torch.empty(mcfg.batch + 1, dtype=torch.int64, device=dev)
        mmap = torch.empty(mb.rows, dtype=torch.int32, device=dev)
        res = {}
        for chunk in (0, 1024):
            ts = []
            for it in range(max(3, args.warmup) + 20):
                flush.fill_(1)
                flush_sum.copy_(flush.view(torch.int64).sum())
                e = new_events(stream, 2)
                e[0].record(stream)
                mpm.merge(mx, moff, workspace=mws, out_tokens=mout, out_offsets=moo, out_map=mmap, chunk=chunk)
                e[1].record(stream)
                if it >= max(3, args.warmup):
                    torch.cuda.synchronize(dev)
                    ts.append(1e3 * e[0].elapsed_time(e[1]))
            res[chunk] = (statistics.median(ts), int(moo[-1]))
        chunked = {
            "workload": mcfg.description, "tokens": mb.rows,
            "merge_us_full": res[0][0], "merge_us_chunk_1024": res[1024][0],
            "speedup": res[0][0] / res[1024][0],
            "merged_tokens_full": res[0][1], "merged_tokens_chunk_1024": res[1024][1],
        }

    # ---------------- fp32 tokens: three tf32 products on the tensor cores vs CUDA-core FMA ----------------
    # The nearest-neighbour step (Eq. 1 + arg max) of the same image shapes
    # in fp32, through MPM_NN_TCGEN05_PAIR (the fp32 default) and MPM_NN_SIMT.
    fp32 = None
    if rank == 0 and not args.no_fp32:
        f_cfg = WorkloadConfig("vit_b_fp32", cfg.batch, cfg.sides, cfg.dim, "f32", cfg.k_range, cfg.sigma_range,
                               cfg.insertions, cfg.seed)
        fb = make_batch(f_cfg)
        fx = fb.tokens.to(dev)
        foff = torch.from_numpy(fb.offsets).to(dev)
        fws = mpm.new_workspace(fb.rows, f_cfg.batch, f_cfg.dim, fx.dtype, dev)
        f_us, f_nn = {}, {}
        for algo in ("tcgen05_pair", "simt"):
            ts = []
            for it in range(max(3, args.warmup) + 10):
                flush.fill_(1)
                flush_sum.copy_(flush.view(torch.int64).sum())
                e = new_events(stream, 2)
                e[0].record(stream)
                nn_f, _ = mpm.nearest_neighbors(fx, foff, algo=algo, workspace=fws, with_score=False)
                e[1].record(stream)
                if it >= max(3, args.warmup):
                    torch.cuda.synchronize(dev)
                    ts.append(1e3 * e[0].elapsed_time(e[1]))
            f_us[algo] = statistics.median(ts)
            f_nn[algo] = nn_f
        fp32 = {
            "workload": f"{f_cfg.batch} x {int(fb.offsets[1])} tokens x {f_cfg.dim} fp32 (vit_b shapes)",
            "nn_us_tensor_3xtf32": f_us["tcgen05_pair"], "nn_us_simt_fma": f_us["simt"],
            "speedup": f_us["simt"] / f_us["tcgen05_pair"],
            "same_neighbour_frac": float((f_nn["tcgen05_pair"] == f_nn["simt"]).float().mean()),
        }

    # ---------------- end to end: host buffers, copies inside the timed region ----------------
    # A serving loop: every step copies its tokens and offsets in from pinned
    # host memory, runs the whole step (L2 flush, merge, stand-in noise,
    # merge, compose, gather) and copies the reconstructed grid back out.
    # Three streams overlap step k's compute with step k+1's copy in and
    # step k-1's copy out (inputs and outputs double-buffered; the host link
    # carries both directions at once).  Timed from the first copy in to the
    # last copy out, everything inside: value = images / that time.
    e2e = None
    if not args.no_e2e:
        host_x = batch.tokens.pin_memory()
        host_off = torch.from_numpy(batch.offsets).pin_memory()
        host_up = [torch.empty(up.shape, dtype=up.dtype).pin_memory() for _ in range(2)]
        dev_x = [x0, torch.empty_like(x0)]
        dev_off = [off0, torch.empty_like(off0)]
        dev_up = [up, torch.empty_like(up)]
        s_in, s_out = torch.cuda.Stream(dev), torch.cuda.Stream(dev)
        inputs_free = [torch.cuda.Event() for _ in range(2)]   # compute finished reading slot s
        inputs_ready = [torch.cuda.Event() for _ in range(2)]  # copy in of slot s landed
        output_ready = [torch.cuda.Event() for _ in range(2)]  # grid of slot s computed
        output_free = [torch.cuda.Event() for _ in range(2)]   # copy out of slot s finished
        for e in inputs_free + output_free:
            e.record(stream)

        def pipelined(n_steps):
            for k in range(n_steps):
                sl = k % 2
                with torch.cuda.stream(s_in):
                    s_in.wait_event(inputs_free[sl])
                    dev_x[sl].copy_(host_x, non_blocking=True)
                    dev_off[sl].copy_(host_off, non_blocking=True)
                    inputs_ready[sl].record(s_in)
                stream.wait_event(inputs_ready[sl])
                stream.wait_event(output_free[sl])
                flush.fill_(1)
                flush_sum.copy_(flush.view(torch.int64).sum())
                mpm.merge(dev_x[sl], dev_off[sl], workspace=ws, out_tokens=x1, out_offsets=off1, out_map=m1)
                if two:
                    x1n[:t1] = apply_noise(x1[:t1], noise)
                    mpm.merge(x1n, off1, workspace=ws, out_tokens=x2, out_offsets=off2, out_map=m2)
                    mpm.compose_gather(x2, off2, m1, dev_off[sl], m2, off1, out=dev_up[sl], out_map=rstar)
                else:
                    mpm.unmerge_gather(x1, off1, m1, dev_off[sl], out=dev_up[sl])
                inputs_free[sl].record(stream)
                output_ready[sl].record(stream)
                with torch.cuda.stream(s_out):
                    s_out.wait_event(output_ready[sl])
                    host_up[sl].copy_(dev_up[sl], non_blocking=True)
                    output_free[sl].record(s_out)

        pipelined(max(2, args.warmup))
        barrier()
        t_start, t_end = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        t_start.record(s_in)
        s_in.wait_event(t_start)
        pipelined(args.steps)
        s_out.wait_stream(stream)
        s_out.wait_stream(s_in)
        t_end.record(s_out)
        barrier()
        e_ms = max_over_ranks(t_start.elapsed_time(t_end) / args.steps)
        # The copied-back grids must be the device result.
        for sl in range(2):
            assert torch.equal(host_up[sl].to(dev), up), "copied-back grid differs from the device result"
        e2e = {"value": global_images / (e_ms * 1e-3), "unit": UNIT,
               "h2d_bytes_per_step": int(host_x.numel() * host_x.element_size() + host_off.numel() * 8),
               "d2h_bytes_per_step": int(host_up[0].numel() * host_up[0].element_size()),
               "ms_per_step": e_ms,
               "pipeline": "3 streams: copy in of step k+1 and copy out of step k-1 overlap step k; "
                           "timed from the first copy in to the last copy out"}

    # The same step on the traced library, in a child process: each kernel's
    # duration inside the step (device timer), next to the CUDA-event figures
    # above, which add launch latency.  roofline.achieved stays the event one.
    in_step = None
    if rank == 0 and world == 1 and not args.no_timeline:
        in_step = in_step_timeline(args.workload)

    if world > 1:
        dist.barrier()
    if rank == 0:
        line = {
            "metric": METRIC, "value": global_images / (ms * 1e-3), "unit": UNIT, "n_gpus": world,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms, "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": cfg.dtype, "data": "synthetic",
            "config": workload_desc(cfg, batch, world),
            "tokens_per_s": float(sum(sizes)) / (ms * 1e-3),
            "merged_tokens": {"stage0": int(n0.sum()), "stage1": int(n1.sum()), "stage2": int(n2.sum())},
            "roofline": roofline,
            "hbm_kernels": hbm_kernels,
            "pipeline_roofline": m["pipeline"],
            "per_workload": per_workload,
            "padded_batch": padded,
            "chunked_similarity": chunked,
            "fp32_nearest_neighbours": fp32,
            "kernels_us": kern,
            "ms_per_step_with_kernel_events": ms_with_kernel_events,
            "in_step": in_step,
            "cpu_baseline": cpu_base,
            "e2e": e2e,
            "clocks": clk,
            "gpu_launches": p.launches() * args.steps,
            "wall_s_timed_loop": wall,
        }
        print(json.dumps(line), flush=True)
    if world > 1:
        dist.destroy_process_group()
    return 0


# ---------------------------------------------------------------------------
# Device timeline of the step (traced library)
# ---------------------------------------------------------------------------
def in_step_timeline(workload):
    """Runs `bench.py --timeline` for `workload` in a child process (one MPM
    library per process) and condenses its line; None if it fails."""
    import subprocess

    cmd = [sys.executable, os.path.abspath(__file__), "--timeline", "--workload", workload, "--steps", "10",
           "--warmup", "3"]
    try:
        res = subprocess.run(cmd, capture_output=True, text=True, timeout=600, cwd=ROOT)
        tl = json.loads(res.stdout.strip().splitlines()[-1])["timeline"]
    except (subprocess.SubprocessError, OSError, ValueError, IndexError, KeyError):
        return None
    aff = [k for k in ("affinity_1", "affinity_2") if k in tl]
    us = sum(tl[k]["us_after_wait"] for k in aff)
    tflop = sum(tl[k]["tflops_algorithmic"] * tl[k]["us_after_wait"] * 1e-6 for k in aff)
    peaks, _ = load_peaks()
    tf = tflop / (us * 1e-6)
    return {
        "source": "python bench.py --timeline --steps 10 --warmup 3 (traced library, GPU global timer, medians)",
        "kernels_us": {k: v["us_after_wait"] for k, v in tl.items()},
        "affinity_tflops_algorithmic": tf,
        "affinity_frac_of_sustained_bf16": tf / peaks.get("bf16_tflops_sustained",
                                                            FALLBACK_PEAKS["bf16_tflops_sustained"]),
        "hbm_gbs": {k: v["gbs"] for k, v in tl.items() if "gbs" in v},
    }


def run_timeline(args):
    """The benchmark step with the device timeline of libmpm_trace.so: for
    every kernel, the time from the moment its blocks passed their wait for
    the previous kernel to its last warp's end (GPU global timer), and the gap
    since the previous kernel ended.  Inside the step, without the CUDA events
    between kernels that the per-kernel figures of the benchmark need."""
    import torch

    import paper_2604_05718_gb300 as mpm
    from paper_2604_05718_gb300 import build
    from workloads import CONFIGS, apply_noise, make_batch, stage_noise

    _, world, _ = dist_env()
    if world > 1:
        raise RuntimeError("--timeline runs on one GPU")
    dev = torch.device("cuda", 0)
    torch.cuda.set_device(dev)
    mpm.library(build.build(trace=True))
    cfg = CONFIGS[args.workload]
    batch = make_batch(cfg)
    dim, esize = cfg.dim, (2 if cfg.dtype == "bf16" else 4)
    two = cfg.insertions == 2
    x0 = batch.tokens.to(dev)
    off0 = torch.from_numpy(batch.offsets).to(dev)
    ws = mpm.new_workspace(batch.rows, cfg.batch, dim, x0.dtype, dev)
    x1, off1, m1 = mpm.merge(x0, off0, workspace=ws)
    off1_h = off1.cpu().numpy()
    t1 = int(off1_h[-1])
    noise = stage_noise(cfg.seed, np.diff(off1_h).tolist(), dim).to(dev) if two else None
    x1n = torch.zeros_like(x1)
    flush = torch.empty(L2_FLUSH_BYTES, dtype=torch.uint8, device=dev)
    flush_sum = torch.zeros((), dtype=torch.int64, device=dev)
    rows = {}
    order = []

    def record(stage, tl, prev_end):
        for kind in ("prep", "affinity", "mutual_scan", "pair_average", "gather", "compose"):
            if kind not in tl:
                continue
            start, waited, end = tl[kind]
            key = f"{kind}_{stage}" if kind not in ("gather", "compose") else kind
            if key not in rows:
                rows[key] = []
                order.append(key)
            rows[key].append(((end - waited) * 1e-3, (end - start) * 1e-3,
                              (waited - prev_end) * 1e-3 if prev_end else float("nan")))
            prev_end = end
        return prev_end

    for it in range(args.warmup + args.steps):
        flush.fill_(1)
        flush_sum.copy_(flush.view(torch.int64).sum())
        mpm.trace_reset()
        x1, off1, m1 = mpm.merge(x0, off0, workspace=ws)
        tl1 = mpm.trace_read()
        if two:
            x1n[:t1] = apply_noise(x1[:t1], noise)
            torch.cuda.synchronize(dev)
            mpm.trace_reset()
            x2, off2, m2 = mpm.merge(x1n, off1, workspace=ws)
            mpm.compose_gather(x2, off2, m1, off0, m2, off1)
        else:
            mpm.trace_reset()
            mpm.unmerge_gather(x1, off1, m1, off0)
        tl2 = mpm.trace_read()
        if it >= args.warmup:
            record(1, tl1, 0)
            record(2, tl2, 0)
    n0 = np.diff(batch.offsets).astype(np.float64)
    n1 = np.diff(off1_h).astype(np.float64)
    n2 = np.diff(off2.cpu().numpy()).astype(np.float64) if two else n1
    hbm_bytes = {
        "prep_1": n0.sum() * dim * esize + 12 * n0.sum(),
        "prep_2": n1.sum() * dim * esize + 12 * n1.sum(),
        "pair_average_1": (n0.sum() + n1.sum()) * dim * esize + 12 * n0.sum(),
        "pair_average_2": (n1.sum() + n2.sum()) * dim * esize + 12 * n1.sum(),
        "gather": (n2.sum() + n0.sum()) * dim * esize + (12 if two else 4) * n0.sum(),
    }
    flops = {"affinity_1": float(np.sum(n0 * (n0 - 1) * dim)), "affinity_2": float(np.sum(n1 * (n1 - 1) * dim))}
    peaks, peak_kind = load_peaks()
    out = {}
    for key in order:
        run = np.array(rows[key])
        med = float(np.median(run[:, 0]))
        entry = {"us_after_wait": med, "us_from_first_block": float(np.median(run[:, 1])),
                 "gap_us_after_previous_kernel": float(np.nanmedian(run[:, 2])) if np.isfinite(run[:, 2]).any()
                 else None}
        if key in hbm_bytes:
            gbs = hbm_bytes[key] / (med * 1e-6) / 1e9
            entry.update(gbs=gbs, hbm_frac=gbs / peaks.get("hbm_gbs", FALLBACK_PEAKS["hbm_gbs"]))
        if key in flops:
            tf = flops[key] / (med * 1e-6) / 1e12
            entry.update(tflops_algorithmic=tf,
                         tensor_frac=tf / peaks.get("bf16_tflops_sustained", FALLBACK_PEAKS["bf16_tflops_sustained"]))
        out[key] = entry
    line = {"timeline": out, "workload": workload_desc(cfg, batch)["workload"], "steps": args.steps,
            "warmup": args.warmup, "peaks": peak_kind,
            "method": "GPU global timer in the traced library; L2 flushed before each step; the host reads "
                      "the timeline after each merge, so the two merges do not overlap"}
    print(json.dumps(line), flush=True)
    return 0


def main():
    args = parse_args()
    if args.impl == "reference":
        return run_reference(args)
    if args.timeline:
        return run_timeline(args)
    return run_mpm(args)


if __name__ == "__main__":
    sys.exit(main())
