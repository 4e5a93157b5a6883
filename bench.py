"""Benchmark: ROI-aware multi-sweep LiDAR voxelization on GB300.

One step = one call of the whole path (motion compensation, ROI test, voxel
grouping, cap and canonical order, mean features) over a 32-frame streaming batch
of nuScenes-shaped frames (11,110,400 points, 222 MB of fp32 input), inputs
resident in HBM. The metric is in-ROI points (points passing the range and
ROI tests, counted before the caps) per second, over the whole job.

  python bench.py [--gpus N --steps K --warmup W] [--impl reference]

With N > 1 (torchrun) every rank voxelizes its own 32 frames (distinct seeds,
no collective on the data path) and rank 0 reports the aggregate over the
slowest rank's time ("weak" scaling). ``--impl reference`` times the CPU
oracle on the host cores instead (a bounded sample of the same workload).
"""
from __future__ import annotations

import argparse
import hashlib
import json
import os
import subprocess
import sys
import threading
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

import synth  # noqa: E402

METRIC = "in-ROI LiDAR points voxelized/sec and µs/frame; achieved HBM GB/s vs peak"
FRAMES = 32
BYTES_PER_POINT = 20      # fp32 x, y, z, intensity, dt
BYTES_PER_VOXEL = 36      # 5 fp32 means + 3 int32 coords + 1 int32 count


def dist_env():
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return world, rank, local


def aggregate_ranks(ms_total: float, e2e_s: float, n_points: float, world: int, device):
    """Whole-job figures over the ranks: the slowest rank's times (MAX) and
    the points all ranks processed (SUM). Each rank voxelizes its own frames,
    so this is the only exchange, and it runs outside the timed regions."""
    import torch
    import torch.distributed as dist
    t = torch.tensor([ms_total, e2e_s], dtype=torch.float64, device=device)
    pts = torch.tensor([float(n_points)], dtype=torch.float64, device=device)
    if world > 1:
        dist.all_reduce(t, op=dist.ReduceOp.MAX)
        dist.all_reduce(pts, op=dist.ReduceOp.SUM)
    return float(t[0].item()), float(t[1].item()), float(pts[0].item())


def workload_for_rank(rank: int, frames: int = FRAMES):
    return synth.streaming_batch(frames, base_seed=1000 + FRAMES * rank)


def workload_desc(w):
    return {
        "workload": (f"batch{w.num_frames}: {w.num_frames} independent nuScenes-shaped frames "
                     "(10 sweeps x 34,720 pts, 32-beam spinning LiDAR, ray-cast scene), "
                     "30 rotated ROIs/frame, margin 0.5 m, 0.075x0.075x0.2 m voxels "
                     "(1440x1440x40), K=10, max 120,000 voxels/frame"),
        "frames_per_gpu": w.num_frames,
        "points_per_gpu": w.num_points,
        "input_mb_per_gpu": round(w.points.nbytes / 1e6, 1),
        "l2": ("inputs (222 MB/step) larger than the 129 MB L2, no flush in the timed region; "
               "l2_flushed gives the call after a 258 MB buffer write"),
    }


def sort_passes(dims) -> int:
    """Launches of the sort stage for a grid: one per 9-bit digit of the
    largest linear index."""
    maxlin = int(dims[0]) * int(dims[1]) * int(dims[2]) - 1
    return (maxlin.bit_length() + 8) // 9


def read_peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(path):
        with open(path) as fh:
            j = json.load(fh)
        return float(j["hbm_gbs"]), "measured"
    return 6800.0, "fallback"


# Algorithmic bytes per launch of each stage (the dominant one is reported):
# the classify pass reads every point once (20 B); the whole path also
# writes 36 B per output voxel.
def dominant_bytes(stage, w, n_in_roi, u_out):
    if stage == "classify":
        return BYTES_PER_POINT * w.num_points
    return BYTES_PER_POINT * w.num_points + BYTES_PER_VOXEL * u_out


def profile_traffic(stage):
    """DRAM bytes per launch of the dominant kernel from the committed ncu
    summary (profiles/<stage>_batch32.json), scaled to this workload, or
    None when there is none or the kernel source changed since it was taken."""
    path = os.path.join(ROOT, "profiles", f"{stage}_batch32.json")
    if not os.path.exists(path):
        return None
    with open(path) as fh:
        j = json.load(fh)
    src = os.path.join(ROOT, "paper_2608_15437_gb300", "csrc", j["source"])
    with open(src, "rb") as fh:
        digest = hashlib.sha256(fh.read()).hexdigest()
    if digest != j.get("source_sha256"):
        return None
    return j.get("dram_bytes_per_launch")


class ClockSampler:
    """nvidia-smi samples (every 50 ms) from just before the timed region to
    the end of the per-kernel breakdown run that follows it."""

    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index: int):
        self.gpu = gpu_index
        self.proc = None
        self.lines = []
        self.thread = None

    def start(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--id={self.gpu}", f"--query-gpu={self.FIELDS}",
                 "--format=csv,noheader,nounits", "-lms", "50"],
                stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except OSError:
            self.proc = None
            return
        self.t0 = time.perf_counter()
        self.thread = threading.Thread(target=self._read, daemon=True)
        self.thread.start()

    def _read(self):
        for line in self.proc.stdout:
            self.lines.append(line.strip())

    def mark(self) -> int:
        """Index of the next sample: brackets a window for ``summary``."""
        return len(self.lines)

    def stop(self):
        if self.proc is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
        if self.thread:
            self.thread.join(timeout=2)
        out = self.summary(0, len(self.lines))
        out["window_s"] = round(time.perf_counter() - self.t0, 3)
        return out

    def summary(self, i0: int, i1: int):
        """Median SM clock, max clock and throttle reasons of samples [i0, i1)."""
        sm, smax, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for ln in self.lines[i0:i1]:
            parts = [x.strip() for x in ln.split(",")]
            if len(parts) < 9:
                continue
            try:
                sm.append(float(parts[1]))
                smax.append(float(parts[2]))
            except ValueError:
                continue
            for name, v in zip(names, parts[5:9]):
                if v.lower().startswith("active"):
                    reasons.add(name)
        return {"sm_mhz": float(np.median(sm)) if sm else None,
                "sm_max_mhz": float(max(smax)) if smax else None,
                "samples": len(sm), "reasons": sorted(reasons)}


def cpu_model() -> str:
    """The host CPU's model name (lscpu, else /proc/cpuinfo)."""
    try:
        out = subprocess.run(["lscpu"], capture_output=True, text=True, timeout=10).stdout
        for ln in out.splitlines():
            if ln.strip().lower().startswith("model name"):
                return ln.split(":", 1)[1].strip()
    except (OSError, subprocess.SubprocessError):
        pass
    try:
        with open("/proc/cpuinfo") as fh:
            for ln in fh:
                if ln.lower().startswith(("model name", "cpu model")):
                    return ln.split(":", 1)[1].strip()
    except OSError:
        pass
    return "unknown"


class PinnedToOneCore:
    """Run the enclosed block on one host core (the last one this process may
    use), then restore the process's affinity."""

    def __enter__(self):
        self.saved = None
        self.core = None
        if hasattr(os, "sched_getaffinity"):
            self.saved = os.sched_getaffinity(0)
            self.core = max(self.saved)
            os.sched_setaffinity(0, {self.core})
        return self

    def __exit__(self, *exc):
        if self.saved is not None:
            os.sched_setaffinity(0, self.saved)
        return False


def host_desc(pin):
    return {"nproc": os.cpu_count(),
            "allowed_cores": (len(pin.saved) if pin.saved is not None else None),
            "pinned_core": pin.core, "cpu_model": cpu_model()}


def cpu_oracle_baseline(w, budget_s: float = 12.0):
    """The oracle as it stands, single-threaded and pinned to one host core,
    on whole frames of the same batch until about budget_s seconds have run."""
    import oracle
    oracle.build()
    frames = 0
    f = 0
    with PinnedToOneCore() as pin:
        t0 = time.perf_counter()
        while True:
            fw = w.frame(f % w.num_frames)
            oracle.voxelize_roi(fw.points, fw.sweep_offsets, fw.sweep_tf, fw.rois, fw.roi_margin,
                                fw.voxel_size, fw.pc_range, fw.max_pts_per_voxel, fw.max_voxels)
            frames += 1
            f += 1
            if time.perf_counter() - t0 >= budget_s:
                break
        dt = time.perf_counter() - t0
    return frames, dt, host_desc(pin)


def run_reference(args):
    world, rank, _ = dist_env()
    if rank != 0:
        return 0
    import oracle
    oracle.build()
    w = workload_for_rank(0)
    per_step = 1  # frames per step: a bounded sample of the batch
    frames = [w.frame(f) for f in range(w.num_frames)]
    in_roi = []
    for fw in frames:  # the metric's numerator per frame, untimed
        _, lin, _ = oracle.classify(fw.points, fw.sweep_offsets, fw.sweep_tf, fw.rois,
                                    fw.roi_margin, fw.voxel_size, fw.pc_range)
        in_roi.append(int((lin >= 0).sum()))
    pts_done = 0
    times = []
    f = 0
    with PinnedToOneCore() as pin:
        for step in range(args.warmup + args.steps):
            t0 = time.perf_counter()
            npts = 0
            for _ in range(per_step):
                fw = frames[f % len(frames)]
                oracle.voxelize_roi(fw.points, fw.sweep_offsets, fw.sweep_tf, fw.rois,
                                    fw.roi_margin, fw.voxel_size, fw.pc_range,
                                    fw.max_pts_per_voxel, fw.max_voxels)
                npts += in_roi[f % len(frames)]
                f += 1
            dt = time.perf_counter() - t0
            if step >= args.warmup:
                times.append(dt)
                pts_done += npts
    total = sum(times)
    value = pts_done / total
    line = {
        "impl": "reference", "metric": METRIC, "value": value, "unit": "points/s",
        "n_gpus": args.gpus, "steps": args.steps, "warmup": args.warmup,
        "ms_per_step": 1e3 * total / len(times), "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "f32", "data": "synthetic",
        "config": workload_desc(w),
        "cpu_baseline": {"kind": "oracle", "value": value, "unit": "points/s", "cores": 1,
                         "sample": f"{per_step} whole frames of the batch per step, "
                                   "single-threaded C oracle pinned to one core",
                         **host_desc(pin)},
        "e2e": {"value": value, "unit": "points/s", "h2d_bytes_per_step": 0,
                "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)
    return 0


def run_gpu(args):
    import torch
    import torch.distributed as dist

    import paper_2608_15437_gb300 as mmbev

    world, rank, local = dist_env()
    if world > 1:
        torch.cuda.set_device(local)
        dist.init_process_group("nccl", device_id=torch.device("cuda", local))
    dev = torch.device("cuda", local if world > 1 else 0)
    mmbev.load()

    w = workload_for_rank(rank, args.frames)
    if args.pillars:   # the same frames on a pillar grid (nz = 1)
        w.voxel_size = np.array([0.075, 0.075, 8.0], np.float32)
    pts = torch.from_numpy(w.points).to(dev)
    tf = torch.from_numpy(w.sweep_tf).to(dev)
    rois = torch.from_numpy(w.rois).to(dev)
    rmax = int(np.max(np.diff(w.frame_roi_offsets)))
    vx = mmbev.Voxelizer(w.num_points, rmax, w.max_voxels, w.num_frames, w.voxel_size,
                         w.pc_range, w.max_pts_per_voxel, w.roi_margin, device=dev,
                         rho_out=args.rho_out, seed=args.seed)
    stream = torch.cuda.current_stream(dev)
    nstage = mmbev.NUM_STAGES
    # ScatterToBEV (Alg. 1, last step), part of the step with --bev
    dims = [int(round((float(w.pc_range[a + 3]) - float(w.pc_range[a])) / float(w.voxel_size[a])))
            for a in range(3)]
    canvas = (torch.empty((w.num_frames, dims[2] * 5, dims[1], dims[0]), dtype=torch.float32,
                          device=dev) if args.bev else None)

    # Temporal ROIs (Sec. IV-C), part of the step with --build-rois: every
    # frame's ROI boxes become previous-frame objects with seeded velocities,
    # and the device builds the ranked table the call then uses
    crit = dict(v_ego=10.0, dt=0.1, a_brake=6.0, d_min=10.0, theta_max_deg=60.0,
                theta_min_deg=15.0, v_wide=5.0, v_narrow=30.0, tau_vru=1.5, tau_motor=2.5,
                r_coll=2.0)
    roi_off = w.frame_roi_offsets
    objs_d = None
    if args.build_rois:
        orng = np.random.default_rng(4242 + rank)
        objs = np.zeros((w.rois.shape[0], 8), np.float32)
        objs[:, :5] = w.rois
        objs[:, 5] = orng.uniform(-5, 20, len(objs))
        objs[:, 6] = orng.uniform(-3, 3, len(objs))
        objs[:, 7] = orng.integers(0, 3, len(objs))
        objs_d = mmbev.pack_objects(torch.from_numpy(objs).to(dev))
        rois_buf = (torch.empty((2 * len(objs), 5), dtype=torch.float32, device=dev),
                    torch.empty(len(objs), dtype=torch.int32, device=dev))
        obj_off = np.asarray(w.frame_roi_offsets, np.int32)
        roi_off = (2 * obj_off).astype(np.int32)
        rmax = 2 * rmax
        vx = mmbev.Voxelizer(w.num_points, rmax, w.max_voxels, w.num_frames, w.voxel_size,
                             w.pc_range, w.max_pts_per_voxel, w.roi_margin, device=dev,
                             rho_out=args.rho_out, seed=args.seed)

    # the metric's numerator: in-ROI points, counted by the library's own
    # per-point classification of these inputs (S1-S2) with the ROI table the
    # step uses, once, untimed
    rois_used = rois if objs_d is None else mmbev.build_rois(objs_d, obj_off, crit)[0]
    _, lin, _ = mmbev.classify_points(pts, w.sweep_offsets, tf, rois_used, w.roi_margin,
                                      w.voxel_size, w.pc_range, w.frame_sweep_offsets, roi_off,
                                      workspace=vx.workspace)
    n_in_roi = int((lin >= 0).sum().item())
    del lin

    # with --bev the outputs are double-buffered, so each step's scatter only
    # clears the previous step's cells (the canvas then equals a full fill
    # and scatter of the step's outputs)
    bev_outs = [vx.out, mmbev.Outputs.empty(w.num_frames, w.max_voxels, dev)] if args.bev else None
    bev_prev = [None]

    def step(**kw):
        rl = rois
        if objs_d is not None:
            rl = mmbev.build_rois(objs_d, obj_off, crit, out=rois_buf)[0]
        if canvas is not None:
            vx.out = bev_outs[1] if vx.out is bev_outs[0] else bev_outs[0]
        out = vx(pts, w.sweep_offsets, tf, rl, w.frame_sweep_offsets, roi_off, **kw)
        if canvas is not None:
            if bev_prev[0] is None or args.bev_full:
                mmbev.scatter_bev(out, w.max_voxels, dims, canvas=canvas)
            else:
                mmbev.scatter_bev_update(bev_prev[0], out, w.max_voxels, dims, canvas)
            bev_prev[0] = out
        return out
    step_ev = [[torch.cuda.Event(enable_timing=True) for _ in range(nstage + 1)]
               for _ in range(args.steps)]
    for evs in step_ev:
        for e in evs:
            e.record(stream)  # materialise the events before handing them to the library
    for _ in range(args.warmup):
        step()
    torch.cuda.synchronize(dev)
    status = vx.status()
    if status != 0:
        raise RuntimeError(f"device status {status:#x} after warm-up")
    nvox = vx.out.nvox.cpu().numpy()
    u_out = int(nvox.sum())

    sampler = ClockSampler(dev.index if dev.index is not None else 0)
    sampler.start()
    time.sleep(0.1)
    start = torch.cuda.Event(enable_timing=True)
    end = torch.cuda.Event(enable_timing=True)
    # timed region 1, the headline: K back-to-back calls, kernels chained by
    # programmatic dependent launch
    if world > 1:
        dist.barrier()
    torch.cuda.synchronize(dev)
    start.record(stream)
    for k in range(args.steps):
        step()
    end.record(stream)
    torch.cuda.synchronize(dev)
    if world > 1:
        dist.barrier()
    ms_total = start.elapsed_time(end)
    i_timed = sampler.mark()
    # a sustained window of the same calls, about a second and a half long, so
    # that the clock samples (every 50 ms) describe the clock the calls ran at
    n_sus = max(args.steps, int(1500.0 / max(ms_total / args.steps, 1e-3)))
    i_sus = sampler.mark()
    start.record(stream)
    for k in range(n_sus):
        step()
    end.record(stream)
    torch.cuda.synchronize(dev)
    sus_ms = start.elapsed_time(end)
    i_sus_end = sampler.mark()
    sus_clock = sampler.summary(i_sus, i_sus_end)
    sus_us = 1e3 * sus_ms / n_sus
    sustained = {"calls": n_sus, "us_per_call": round(sus_us, 2), **sus_clock,
                 "us_x_mhz": (round(sus_us * sus_clock["sm_mhz"], 1)
                              if sus_clock.get("sm_mhz") else None)}
    # each call after a write of a buffer twice the size of L2: nothing the
    # previous call left in L2 (lists, counters, outputs) survives
    flush = torch.empty(2 * 129 * 2**20 // 4, dtype=torch.float32, device=dev)
    n_fl = max(3, min(args.steps, 50))
    fl_ms = 0.0
    for k in range(n_fl):
        flush.fill_(float(k))
        start.record(stream)
        step()
        end.record(stream)
        torch.cuda.synchronize(dev)
        fl_ms += start.elapsed_time(end)
    del flush
    l2_flushed = {"calls": n_fl, "us_per_call": round(1e3 * fl_ms / n_fl, 2)}
    # timed region 2, the per-kernel breakdown: the same K calls with a CUDA
    # event on the launching stream between consecutive kernels
    for k in range(args.steps):
        step(stage_events=step_ev[k])
    torch.cuda.synchronize(dev)
    rois_us = None
    if objs_d is not None:   # the ROI construction alone
        r0e = torch.cuda.Event(enable_timing=True)
        r1e = torch.cuda.Event(enable_timing=True)
        r0e.record(stream)
        for k in range(args.steps):
            mmbev.build_rois(objs_d, obj_off, crit, out=rois_buf)
        r1e.record(stream)
        torch.cuda.synchronize(dev)
        rois_us = 1e3 * r0e.elapsed_time(r1e) / args.steps
    cc_us = cc_n = None
    if args.components:   # the voxel-grid proposer alone, on the last call's outputs
        need = mmbev.components_table_bytes(w.num_frames, w.max_voxels)
        cc_table = torch.zeros(need, dtype=torch.uint8, device=dev) if need else None
        c0e = torch.cuda.Event(enable_timing=True)
        c1e = torch.cuda.Event(enable_timing=True)
        c0e.record(stream)
        for k in range(args.steps):
            cc = mmbev.voxel_components(vx.out, w.max_voxels, dims, cc_table)
        c1e.record(stream)
        torch.cuda.synchronize(dev)
        cc_us = 1e3 * c0e.elapsed_time(c1e) / args.steps
        cc_n = int(cc[2].sum().item())
    bev_us = bev_upd_us = None
    if canvas is not None:   # ScatterToBEV alone, on the last calls' outputs
        b0 = torch.cuda.Event(enable_timing=True)
        b1 = torch.cuda.Event(enable_timing=True)
        b0.record(stream)
        for k in range(args.steps):
            mmbev.scatter_bev(vx.out, w.max_voxels, dims, canvas=canvas)
        b1.record(stream)
        torch.cuda.synchronize(dev)
        bev_us = 1e3 * b0.elapsed_time(b1) / args.steps
        b0.record(stream)   # the update form, alternating the two output buffers
        for k in range(args.steps):
            mmbev.scatter_bev_update(bev_outs[k % 2], bev_outs[(k + 1) % 2], w.max_voxels, dims,
                                     canvas)
        b1.record(stream)
        torch.cuda.synchronize(dev)
        bev_upd_us = 1e3 * b0.elapsed_time(b1) / args.steps
    clocks_all = sampler.stop()
    # the clocks of the timed region and the sustained window that follows it
    clocks = sampler.summary(0, i_sus_end)
    clocks["window_s"] = clocks_all.get("window_s")
    status = vx.status()
    if status != 0:
        raise RuntimeError(f"device status {status:#x} after the timed steps")

    stage_ms = np.zeros(nstage)
    for evs in step_ev:
        for s in range(nstage):
            stage_ms[s] += evs[s].elapsed_time(evs[s + 1])
    stage_ms /= args.steps
    names = mmbev.stage_names()


    # end to end through the public API: pinned host inputs, H2D, the call,
    # then every frame's kept rows packed by the device straight into a
    # pinned host buffer (offsets and 36-byte records), and one sync
    h_pts = torch.from_numpy(w.points).pin_memory()
    h_tf = torch.from_numpy(w.sweep_tf).pin_memory()
    h_rois = torch.from_numpy(w.rois).pin_memory()
    d_pts = torch.empty_like(pts)
    d_tf = torch.empty_like(tf)
    d_rois = torch.empty_like(rois)
    # two pinned result buffers: the host reads step i's result while step
    # i+1 is in flight (its uploads overlap step i's tail)
    h_packed = [torch.empty(mmbev.pack_bytes(w.num_frames, w.max_voxels),
                            dtype=torch.uint8).pin_memory() for _ in range(2)]
    e2e_steps = max(3, min(args.steps, 10))
    d2h_bytes = 0

    h_objs = objs_d.cpu().pin_memory() if objs_d is not None else None   # packed layout
    d_objs = torch.empty_like(objs_d) if objs_d is not None else None

    def e2e_launch(i):
        dst = h_packed[i % 2]
        if d_objs is None:   # host inputs: chunks go up while earlier ones are voxelized
            out = vx.run_host(h_pts, w.sweep_offsets, h_tf, h_rois, w.frame_sweep_offsets,
                              roi_off, chunk_frames=args.e2e_chunk, pack_dst=dst)
        else:   # the previous frame's objects go up; the ROI table is built on the device
            d_pts.copy_(h_pts, non_blocking=True)
            d_tf.copy_(h_tf, non_blocking=True)
            d_objs.copy_(h_objs, non_blocking=True)
            rl = mmbev.build_rois(d_objs, obj_off, crit, out=rois_buf)[0]
            out = vx(d_pts, w.sweep_offsets, d_tf, rl, w.frame_sweep_offsets, roi_off)
            mmbev.pack_voxels(out, w.max_voxels, dst)
        ev = torch.cuda.Event()
        ev.record(torch.cuda.current_stream(dev))
        return ev

    def e2e_read(i, ev):   # the step's result, on the host
        nonlocal d2h_bytes
        ev.synchronize()
        dst = h_packed[i % 2]
        total = int(dst[4 * w.num_frames:4 * w.num_frames + 4].view(torch.int32)[0])
        d2h_bytes = 4 * (w.num_frames + 1) + BYTES_PER_VOXEL * total

    def e2e_run(n):
        pending = None
        for i in range(n):
            ev = e2e_launch(i)
            if pending is not None:
                e2e_read(*pending)
            pending = (i, ev)
        e2e_read(*pending)

    e2e_run(2)
    if world > 1:
        dist.barrier()
    torch.cuda.synchronize(dev)
    t0 = time.perf_counter()
    e2e_run(e2e_steps)
    torch.cuda.synchronize(dev)
    e2e_local = time.perf_counter() - t0
    # slowest rank decides
    ms_max, e2e_max, total_pts = aggregate_ranks(ms_total, e2e_local, n_in_roi, world, dev)
    ms_step = ms_max / args.steps
    value = total_pts / (ms_step * 1e-3)
    e2e_value = total_pts / (e2e_max / e2e_steps)
    h2d_bytes = w.points.nbytes + w.sweep_tf.nbytes + (
        w.rois.nbytes if objs_d is None else objs.nbytes)

    if rank == 0:
        peak, peak_kind = read_peaks()
        dom = int(np.argmax(stage_ms))
        t_dom = stage_ms[dom] * 1e-3
        achieved = dominant_bytes(names[dom], w, n_in_roi, u_out) / t_dom / 1e9
        path_bytes = BYTES_PER_POINT * w.num_points + BYTES_PER_VOXEL * u_out
        line = {
            "metric": METRIC, "value": value, "unit": "points/s", "n_gpus": world,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms_step,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f32",
            "data": "synthetic", "config": workload_desc(w),
            "us_per_frame": 1e3 * ms_step / w.num_frames,
            "in_roi_points_per_gpu": n_in_roi, "voxels_out_per_gpu": u_out,
            "rho_out": args.rho_out,
            "grid": dims,
            "components": (None if cc_us is None else {"us": round(cc_us, 2), "components": cc_n}),
            "build_rois": (None if rois_us is None else
                           {"us": round(rois_us, 2), "objects": int(objs_d.shape[0])}),
            "scatter_bev": (None if bev_us is None else
                            {"us": round(bev_us, 2), "canvas_mb": round(canvas.numel() * 4 / 1e6, 1),
                             "canvas_gbs": round(canvas.numel() * 4 / (bev_us * 1e-6) / 1e9, 1),
                             "update_us": round(bev_upd_us, 2),
                             "in_step": "full" if args.bev_full else "update"}),
            "path_hbm_gbs": path_bytes / (ms_step * 1e-3) / 1e9,
            "path_frac_of_peak": path_bytes / (ms_step * 1e-3) / 1e9 / peak,
            "stage_us": {n: round(1e3 * t, 2) for n, t in zip(names, stage_ms)},
            "roofline": {"bound": "hbm", "kernel": names[dom], "achieved": achieved,
                         "peak": peak, "peak_kind": peak_kind, "unit": "GB/s",
                         "frac": achieved / peak, "traffic": profile_traffic(names[dom])},
            "stage_sum_us": round(1e3 * float(stage_ms.sum()), 2),
            "clocks": clocks,
            "sustained": sustained,
            "l2_flushed": l2_flushed,
            "e2e": {"value": e2e_value, "unit": "points/s", "h2d_bytes_per_step": h2d_bytes,
                    "d2h_bytes_per_step": d2h_bytes, "steps": e2e_steps},
            # one launch a stage, but one a 9-bit digit of the lins for the sort
            "gpu_launches": (nstage - 1 + sort_passes(dims)) * args.steps,
        }
        if world == 1 and not args.no_small_configs:
            # the single-frame configs (L2-resident, latency-bound): warm us
            # per call, eager and replayed from a CUDA graph
            line["single_frame_configs"] = small_config_rows(args, dev)
        frames, secs, host = cpu_oracle_baseline(w)
        pts_per_frame = n_in_roi / w.num_frames
        line["cpu_baseline"] = {
            "kind": "oracle", "value": frames * pts_per_frame / secs, "unit": "points/s",
            "cores": 1, "sample": f"{frames} whole frames of this batch, single-threaded C "
                                  f"oracle pinned to one core, {secs:.1f} s", **host}
        print(json.dumps(line), flush=True)
    if world > 1:
        dist.destroy_process_group()
    return 0


SMALL_CONFIGS = ("tiny", "nuscenes", "ouster", "roi_0", "roi_8", "roi_32", "roi_128", "roi_full")


def small_config_rows(args, dev):
    """The single-frame configs (tiny, nuScenes- and Ouster-shaped, the ROI
    coverage sweep): L2-resident, so reported as warm us per call, eager and
    replayed from a CUDA graph, with no roofline claim."""
    import torch

    import paper_2608_15437_gb300 as mmbev

    rows = {}
    for name in SMALL_CONFIGS:
        w = synth.CONFIGS[name]()
        pts = torch.from_numpy(w.points).to(dev)
        tf = torch.from_numpy(w.sweep_tf).to(dev)
        rois = torch.from_numpy(np.ascontiguousarray(w.rois, np.float32).reshape(-1, 5)).to(dev)
        rmax = max(1, int(np.max(np.diff(w.frame_roi_offsets))))
        vx = mmbev.Voxelizer(w.num_points, rmax, w.max_voxels, w.num_frames, w.voxel_size,
                             w.pc_range, w.max_pts_per_voxel, w.roi_margin, device=dev)

        def call():
            return vx(pts, w.sweep_offsets, tf, rois, w.frame_sweep_offsets, w.frame_roi_offsets)

        for _ in range(max(3, args.warmup)):
            call()
        torch.cuda.synchronize(dev)
        if vx.status() != 0:
            raise RuntimeError(f"{name}: device status {vx.status():#x}")
        _, lin, _ = mmbev.classify_points(pts, w.sweep_offsets, tf, rois, w.roi_margin,
                                          w.voxel_size, w.pc_range, w.frame_sweep_offsets,
                                          w.frame_roi_offsets, workspace=vx.workspace)
        n_in = int((lin >= 0).sum().item())
        nvox = int(vx.out.nvox.sum().item())
        reps = max(20, min(args.steps, 200))
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record()
        for _ in range(reps):
            call()
        e1.record()
        torch.cuda.synchronize(dev)
        eager = 1e3 * e0.elapsed_time(e1) / reps
        g = torch.cuda.CUDAGraph()
        cs = torch.cuda.Stream(dev)
        with torch.cuda.graph(g, stream=cs):
            call()
        g.replay()
        torch.cuda.synchronize(dev)
        e0.record()
        for _ in range(reps):
            g.replay()
        e1.record()
        torch.cuda.synchronize(dev)
        graph = 1e3 * e0.elapsed_time(e1) / reps
        if vx.status() != 0:
            raise RuntimeError(f"{name}: device status {vx.status():#x}")
        rows[name] = {"points": int(w.num_points), "in_roi_points": n_in, "voxels": nvox,
                      "rois": int(w.rois.reshape(-1, 5).shape[0]), "us_eager": round(eager, 2),
                      "us_graph": round(graph, 2),
                      "kept_fraction": round(n_in / max(int(w.num_points), 1), 4),
                      "in_roi_points_per_s_graph": round(n_in / (graph * 1e-6), 1)}
    return rows


def run_small_configs(args):
    """The single-frame configs alone, as one JSON line."""
    import torch

    import paper_2608_15437_gb300 as mmbev

    dev = torch.device("cuda", 0)
    mmbev.load()
    rows = small_config_rows(args, dev)
    print(json.dumps({"metric": "us per single-frame call (warm; eager and CUDA-graph replay)",
                      "unit": "us", "n_gpus": 1, "data": "synthetic",
                      "higher_is_better": False, "configs": rows}))
    return 0


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=1000)
    ap.add_argument("--warmup", type=int, default=10)
    ap.add_argument("--impl", default="gb300", choices=["gb300", "reference"])
    ap.add_argument("--rho-out", type=float, default=0.0,
                    help="keep probability of points inside no ROI (Alg. 1); the headline "
                         "workload uses 0")
    ap.add_argument("--seed", type=int, default=0, help="seed of the rho_out draws")
    ap.add_argument("--pillars", action="store_true",
                    help="the same frames on a 0.075 x 0.075 x 8 m pillar grid (nz = 1)")
    ap.add_argument("--build-rois", action="store_true",
                    help="build every frame's ROI table on the device from previous-frame "
                         "objects (Sec. IV-C) as part of the step")
    ap.add_argument("--e2e-chunk", type=int, default=8,
                    help="frames per host-to-device chunk in the end-to-end leg")
    ap.add_argument("--components", action="store_true",
                    help="also time the voxel-grid connected-component proposer on the outputs")
    ap.add_argument("--bev", action="store_true",
                    help="add ScatterToBEV (a dense [F, nz*5, ny, nx] canvas) to every step")
    ap.add_argument("--bev-full", action="store_true",
                    help="with --bev: fill the whole canvas every step instead of clearing the "
                         "previous step's cells")
    ap.add_argument("--frames", type=int, default=FRAMES,
                    help="frames per GPU (the headline workload is 32; fewer for small "
                         "profiling cases)")
    ap.add_argument("--no-small-configs", action="store_true",
                    help="leave the single-frame configs out of the headline line")
    ap.add_argument("--small-configs", action="store_true",
                    help="instead of the headline: warm us per call of the single-frame "
                         "configs (tiny, nuScenes, Ouster, ROI sweep)")
    args = ap.parse_args()
    if args.small_configs:
        return run_small_configs(args)
    if args.impl == "reference":
        return run_reference(args)
    return run_gpu(args)


if __name__ == "__main__":
    sys.exit(main())
