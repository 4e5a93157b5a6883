"""Seeded synthetic LiDAR workloads for ROI-aware multi-sweep voxelization.

These generators produce inputs only. They hold none of the voxelization
arithmetic and are shared, read-only, by the oracle tests, the GPU parity
tests and the benchmark. nuScenes and the paper's Ouster drive are not
available, so seeded scenes of the same shape stand in for them:

* ``tiny``: 20,000 uniform points, one sweep, four rotated ROIs, a
  512 x 512 x 1 pillar grid.
* ``nuscenes_frame``: a 32-beam spinning LiDAR (elevations -30..+10 deg,
  1,085 azimuth bins), 10 sweeps with ego motion between them, ray-cast
  against a ground plane at z = -1.8 m and 40 random cuboids; 30 ROIs are
  cuboid footprints; a 1440 x 1440 x 40 grid.
* ``ouster_frame``: 128 beams (-22.5..+22.5 deg) x 1,024 azimuth bins,
  3 sweeps, range capped at 40 m, 16 ROIs with a 1 m margin, 800 x 800 x 30.
* ``roi_coverage``: the nuScenes-shaped scene with 0, 8, 32 or 128 ROIs, or one
  ROI covering the whole range (the dense limit).
* ``streaming_batch``: 32 independent nuScenes-shaped frames in one call.

Points are written in each sweep's own sensor frame; ``sweep_tf[k]`` maps
sweep k into the current frame (rotation about z plus a planar translation),
the transform Eq. 6 applies. Points are ordered azimuth-major (one firing of
all beams, then the next azimuth), as a spinning sensor emits them. A ray that
drops out (5 %) or hits nothing within the sensor's range still yields a point,
placed 1000 m out along the ray with intensity 0, so N is fixed; the range crop
removes it. ROIs are ordered nearest-first as a stand-in for the criticality
ranking of Sec. IV-C, which is upstream of this path.
"""
from __future__ import annotations

from dataclasses import dataclass, field

import numpy as np

GROUND_Z = -1.8
FAR = 1000.0


@dataclass
class Workload:
    """One voxelization call's inputs (host arrays)."""
    name: str
    points: np.ndarray            # float32 [N, 5]: x, y, z, intensity, dt
    sweep_offsets: np.ndarray     # int64 [S + 1]
    sweep_tf: np.ndarray          # float32 [S, 16], row-major 4x4, sweep -> current
    rois: np.ndarray              # float32 [R, 5]: cx, cy, w, l, yaw
    roi_margin: float
    voxel_size: np.ndarray        # float32 [3]
    pc_range: np.ndarray          # float32 [6]: xmin, ymin, zmin, xmax, ymax, zmax
    max_pts_per_voxel: int
    max_voxels: int
    frame_sweep_offsets: np.ndarray = field(default=None)  # int32 [F + 1]
    frame_roi_offsets: np.ndarray = field(default=None)    # int32 [F + 1]

    def __post_init__(self):
        if self.frame_sweep_offsets is None:
            self.frame_sweep_offsets = np.array([0, len(self.sweep_offsets) - 1], np.int32)
        if self.frame_roi_offsets is None:
            self.frame_roi_offsets = np.array([0, self.rois.shape[0]], np.int32)

    @property
    def num_points(self) -> int:
        return int(self.sweep_offsets[-1])

    @property
    def num_frames(self) -> int:
        return len(self.frame_sweep_offsets) - 1

    def frame(self, f: int) -> "Workload":
        """Frame f of a batch as a single-frame workload (indices rebased)."""
        s0, s1 = int(self.frame_sweep_offsets[f]), int(self.frame_sweep_offsets[f + 1])
        r0, r1 = int(self.frame_roi_offsets[f]), int(self.frame_roi_offsets[f + 1])
        p0, p1 = int(self.sweep_offsets[s0]), int(self.sweep_offsets[s1])
        return Workload(
            name=f"{self.name}[{f}]",
            points=self.points[p0:p1].copy(),
            sweep_offsets=(self.sweep_offsets[s0:s1 + 1] - p0).astype(np.int64),
            sweep_tf=self.sweep_tf[s0:s1].copy(),
            rois=self.rois[r0:r1].copy(),
            roi_margin=self.roi_margin,
            voxel_size=self.voxel_size.copy(),
            pc_range=self.pc_range.copy(),
            max_pts_per_voxel=self.max_pts_per_voxel,
            max_voxels=self.max_voxels,
        )

    def with_rois(self, rois: np.ndarray, name: str | None = None, margin=None) -> "Workload":
        """Same single-frame scene with another ROI list."""
        assert self.num_frames == 1
        rois = np.ascontiguousarray(rois, np.float32).reshape(-1, 5)
        return Workload(name=name or self.name, points=self.points,
                        sweep_offsets=self.sweep_offsets, sweep_tf=self.sweep_tf,
                        rois=rois,
                        roi_margin=self.roi_margin if margin is None else float(margin),
                        voxel_size=self.voxel_size, pc_range=self.pc_range,
                        max_pts_per_voxel=self.max_pts_per_voxel,
                        max_voxels=self.max_voxels)


def _pose_matrix(px: float, py: float, yaw: float) -> np.ndarray:
    c, s = np.cos(yaw), np.sin(yaw)
    m = np.array([[c, -s, 0.0, px],
                  [s, c, 0.0, py],
                  [0.0, 0.0, 1.0, 0.0],
                  [0.0, 0.0, 0.0, 1.0]], np.float64)
    return m.astype(np.float32).reshape(16)


def _cuboids(rng: np.random.Generator, n: int, dmin: float = 3.0, dmax: float = 50.0):
    """n static cuboids on the ground: rows (cx, cy, cz, hl, hw, hh, yaw).
    70 % car-like (3.5-5 x 1.6-2 x 1.4-1.8 m), the rest pedestrian-like."""
    d = rng.uniform(dmin, dmax, n)
    ang = rng.uniform(0.0, 2 * np.pi, n)
    car = rng.uniform(0.0, 1.0, n) < 0.7
    l = np.where(car, rng.uniform(3.5, 5.0, n), rng.uniform(0.5, 0.8, n))
    w = np.where(car, rng.uniform(1.6, 2.0, n), rng.uniform(0.5, 0.8, n))
    h = np.where(car, rng.uniform(1.4, 1.8, n), rng.uniform(1.5, 1.9, n))
    yaw = rng.uniform(0.0, 2 * np.pi, n)
    cx, cy = d * np.cos(ang), d * np.sin(ang)
    cz = GROUND_Z + 0.5 * h
    return np.stack([cx, cy, cz, 0.5 * l, 0.5 * w, 0.5 * h, yaw], axis=1)


def _ego_poses(rng: np.random.Generator, n_sweeps: int, step_max: float):
    """Sensor pose (x, y, yaw) of each sweep in the current frame; sweep 0 is
    the current one, older sweeps trail behind by up to step_max per sweep."""
    poses = [(0.0, 0.0, 0.0)]
    for _ in range(1, n_sweeps):
        x, y, th = poses[-1]
        fwd = -rng.uniform(0.0, step_max)
        lat = rng.uniform(-0.1, 0.1)
        dth = rng.uniform(-0.02, 0.02)
        c, s = np.cos(th), np.sin(th)
        poses.append((x + c * fwd - s * lat, y + s * fwd + c * lat, th + dth))
    return poses


def _cast_sweep(rng, dirs_local, az_local, n_beams, pose, boxes, max_range,
                noise_sigma=0.02, dropout=0.05):
    """Ray-cast one sweep from pose against the ground and the cuboids.
    Returns sensor-frame xyz (float64 [M, 3]) and intensity."""
    px, py, yaw = pose
    c, s = np.cos(yaw), np.sin(yaw)
    dw = np.empty_like(dirs_local)
    dw[:, 0] = c * dirs_local[:, 0] - s * dirs_local[:, 1]
    dw[:, 1] = s * dirs_local[:, 0] + c * dirs_local[:, 1]
    dw[:, 2] = dirs_local[:, 2]
    m = dirs_local.shape[0]
    t = np.full(m, np.inf)
    with np.errstate(divide="ignore", invalid="ignore"):
        down = dw[:, 2] < 0
        t[down] = GROUND_Z / dw[down, 2]
    n_az = az_local.shape[0]
    bin_w = 2 * np.pi / n_az
    beams = np.arange(n_beams)
    for b in boxes:
        bx, by, bz, hl, hw, hh, byaw = b
        rx, ry = bx - px, by - py
        dist = np.hypot(rx, ry)
        rho = np.hypot(hl, hw)
        if dist > rho + 1e-3:
            alpha = np.arcsin(min(1.0, rho / dist))
            centre = np.arctan2(ry, rx) - yaw
            diff = np.mod(az_local - centre + np.pi, 2 * np.pi) - np.pi
            a_idx = np.nonzero(np.abs(diff) <= alpha + bin_w)[0]
            if a_idx.size == 0:
                continue
            idx = (a_idx[:, None] * n_beams + beams[None, :]).ravel()
        else:
            idx = np.arange(m)
        cb, sb = np.cos(byaw), np.sin(byaw)
        ox, oy, oz = px - bx, py - by, 0.0 - bz
        o = np.array([cb * ox + sb * oy, -sb * ox + cb * oy, oz])
        d = dw[idx]
        dl = np.stack([cb * d[:, 0] + sb * d[:, 1], -sb * d[:, 0] + cb * d[:, 1], d[:, 2]], 1)
        ext = np.array([hl, hw, hh])
        with np.errstate(divide="ignore", invalid="ignore"):
            t1 = (-ext[None, :] - o[None, :]) / dl
            t2 = (ext[None, :] - o[None, :]) / dl
        tn = np.nanmax(np.minimum(t1, t2), axis=1)
        tf = np.nanmin(np.maximum(t1, t2), axis=1)
        hit = (tn <= tf) & (tn > 0.0)
        sel = idx[hit]
        t[sel] = np.minimum(t[sel], tn[hit])
    t_noisy = t + rng.normal(0.0, noise_sigma, m)
    drop = rng.uniform(0.0, 1.0, m) < dropout
    inten = rng.uniform(0.0, 1.0, m)
    miss = ~np.isfinite(t) | (t > max_range) | drop | (t_noisy <= 0.0)
    r = np.where(miss, FAR, t_noisy)
    inten = np.where(miss, 0.0, inten)
    xyz = dirs_local * r[:, None]
    return xyz, inten


def _spinning_frame(seed, elev_deg, n_az, n_sweeps, sweep_period, max_range,
                    n_rois, step_max=1.5, n_boxes=40):
    """One multi-sweep frame of a spinning LiDAR. Returns points, offsets,
    transforms and nearest-first ROI footprints (w, l from the cuboids)."""
    rng = np.random.default_rng(seed)
    boxes = _cuboids(rng, n_boxes)
    poses = _ego_poses(rng, n_sweeps, step_max)
    el = np.deg2rad(np.asarray(elev_deg, np.float64))
    az = 2 * np.pi * np.arange(n_az) / n_az
    n_beams = el.shape[0]
    ce, se = np.cos(el), np.sin(el)
    dirs = np.stack([np.cos(az)[:, None] * ce[None, :],
                     np.sin(az)[:, None] * ce[None, :],
                     np.broadcast_to(se[None, :], (n_az, n_beams))], axis=2).reshape(-1, 3)
    pts, tfs = [], []
    for k in range(n_sweeps):
        xyz, inten = _cast_sweep(rng, dirs, az, n_beams, poses[k], boxes, max_range)
        p = np.empty((xyz.shape[0], 5), np.float32)
        p[:, :3] = xyz
        p[:, 3] = inten
        p[:, 4] = np.float32(sweep_period * k)
        pts.append(p)
        tfs.append(_pose_matrix(*poses[k]))
    m = n_az * n_beams
    offsets = np.arange(n_sweeps + 1, dtype=np.int64) * m
    pick = rng.permutation(n_boxes)[:n_rois]
    sel = boxes[pick]
    order = np.argsort(np.hypot(sel[:, 0], sel[:, 1]), kind="stable")
    sel = sel[order]
    rois = np.stack([sel[:, 0], sel[:, 1], 2 * sel[:, 4], 2 * sel[:, 3], sel[:, 6]], 1)
    return (np.concatenate(pts, 0), offsets, np.stack(tfs, 0),
            rois.astype(np.float32), boxes)


def tiny(seed: int = 0) -> Workload:
    """20,000 uniform points, 1 sweep, identity transform, 4 rotated ROIs."""
    rng = np.random.default_rng(seed)
    n = 20000
    pts = np.empty((n, 5), np.float32)
    pts[:, 0] = rng.uniform(-51.2, 51.2, n)
    pts[:, 1] = rng.uniform(-51.2, 51.2, n)
    pts[:, 2] = rng.uniform(-5.0, 3.0, n)
    pts[:, 3] = rng.uniform(0.0, 1.0, n)
    pts[:, 4] = 0.0
    rois = np.stack([rng.uniform(-51.2, 51.2, 4), rng.uniform(-51.2, 51.2, 4),
                     rng.uniform(2.0, 6.0, 4), rng.uniform(2.0, 6.0, 4),
                     rng.uniform(0.0, 2 * np.pi, 4)], 1).astype(np.float32)
    return Workload(
        name="tiny", points=pts, sweep_offsets=np.array([0, n], np.int64),
        sweep_tf=np.eye(4, dtype=np.float32).reshape(1, 16), rois=rois, roi_margin=0.5,
        voxel_size=np.array([0.2, 0.2, 8.0], np.float32),
        pc_range=np.array([-51.2, -51.2, -5.0, 51.2, 51.2, 3.0], np.float32),
        max_pts_per_voxel=10, max_voxels=16000)


NUSC_ELEV = np.linspace(-30.0, 10.0, 32)
OUSTER_ELEV = np.linspace(-22.5, 22.5, 128)


def nuscenes_frame(seed: int = 1, n_rois: int = 30) -> Workload:
    """10 sweeps x 34,720 points of a 32-beam spinning LiDAR, 30 ROIs,
    0.075 x 0.075 x 0.2 m voxels over [-54, 54]^2 x [-5, 3]."""
    pts, off, tf, rois, _ = _spinning_frame(seed, NUSC_ELEV, 1085, 10, 0.05, 70.0, n_rois)
    return Workload(
        name="nuscenes", points=pts, sweep_offsets=off, sweep_tf=tf, rois=rois,
        roi_margin=0.5, voxel_size=np.array([0.075, 0.075, 0.2], np.float32),
        pc_range=np.array([-54.0, -54.0, -5.0, 54.0, 54.0, 3.0], np.float32),
        max_pts_per_voxel=10, max_voxels=120000)


def ouster_frame(seed: int = 2) -> Workload:
    """3 sweeps x 131,072 points of a 128-beam sensor capped at 40 m, 16 ROIs
    with a 1 m margin, 0.1 x 0.1 x 0.2 m voxels over [-40, 40]^2 x [-3, 3]."""
    pts, off, tf, rois, _ = _spinning_frame(seed, OUSTER_ELEV, 1024, 3, 0.1, 40.0, 16)
    return Workload(
        name="ouster", points=pts, sweep_offsets=off, sweep_tf=tf, rois=rois,
        roi_margin=1.0, voxel_size=np.array([0.1, 0.1, 0.2], np.float32),
        pc_range=np.array([-40.0, -40.0, -3.0, 40.0, 40.0, 3.0], np.float32),
        max_pts_per_voxel=5, max_voxels=200000)


def roi_coverage(n_rois, scene_seed: int = 1) -> Workload:
    """The nuScenes-shaped scene with n_rois ROIs (seed 10 + n_rois): cuboid
    footprints first, then random boxes; ``n_rois='full'`` gives one
    axis-aligned 1000 x 1000 m ROI covering the whole range."""
    base = nuscenes_frame(scene_seed)
    if n_rois == "full":
        rois = np.array([[0.0, 0.0, 1000.0, 1000.0, 0.0]], np.float32)
        return base.with_rois(rois, name="roi_full")
    n = int(n_rois)
    rng = np.random.default_rng(10 + n)
    boxes = _cuboids(np.random.default_rng(scene_seed), 40)   # the scene's own cuboids
    fp = boxes[rng.permutation(boxes.shape[0])]
    fp = np.stack([fp[:, 0], fp[:, 1], 2 * fp[:, 4], 2 * fp[:, 3], fp[:, 6]], 1)
    k = max(0, n - fp.shape[0])
    extra = np.stack([rng.uniform(-54, 54, k), rng.uniform(-54, 54, k),
                      rng.uniform(1.5, 3.0, k), rng.uniform(2.0, 6.0, k),
                      rng.uniform(0.0, 2 * np.pi, k)], 1)
    rois = np.concatenate([fp[:min(n, fp.shape[0])], extra], 0).astype(np.float32)
    order = np.argsort(np.hypot(rois[:, 0], rois[:, 1]), kind="stable")
    return base.with_rois(rois[order], name=f"roi_{n}")


def concat_frames(frames, name: str) -> Workload:
    """Stack single-frame workloads into one batched call."""
    pts, offs, tfs, rois, fso, fro = [], [0], [], [], [0], [0]
    base = 0
    for w in frames:
        assert w.num_frames == 1
        pts.append(w.points)
        offs.extend((w.sweep_offsets[1:] + base).tolist())
        base += w.num_points
        tfs.append(w.sweep_tf)
        rois.append(w.rois)
        fso.append(fso[-1] + len(w.sweep_offsets) - 1)
        fro.append(fro[-1] + w.rois.shape[0])
    w0 = frames[0]
    return Workload(
        name=name, points=np.concatenate(pts, 0), sweep_offsets=np.array(offs, np.int64),
        sweep_tf=np.concatenate(tfs, 0), rois=np.concatenate(rois, 0).reshape(-1, 5),
        roi_margin=w0.roi_margin, voxel_size=w0.voxel_size, pc_range=w0.pc_range,
        max_pts_per_voxel=w0.max_pts_per_voxel, max_voxels=w0.max_voxels,
        frame_sweep_offsets=np.array(fso, np.int32), frame_roi_offsets=np.array(fro, np.int32))


def streaming_batch(n_frames: int = 32, base_seed: int = 1000) -> Workload:
    """n_frames independent nuScenes-shaped frames (seeds base_seed + f)."""
    frames = [nuscenes_frame(base_seed + f) for f in range(n_frames)]
    return concat_frames(frames, name=f"batch{n_frames}")


CONFIGS = {
    "tiny": tiny,
    "nuscenes": nuscenes_frame,
    "ouster": ouster_frame,
    "roi_0": lambda: roi_coverage(0),
    "roi_8": lambda: roi_coverage(8),
    "roi_32": lambda: roi_coverage(32),
    "roi_128": lambda: roi_coverage(128),
    "roi_full": lambda: roi_coverage("full"),
    "batch32": streaming_batch,
}
