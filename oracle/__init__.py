"""Oracle for ROI-aware multi-sweep LiDAR voxelization (MM-BEV, Sec. IV-D, IV-F).

TEST INFRASTRUCTURE. This package is the plain, slow, single-threaded CPU
statement of the path (motion compensation, Eq. 6-7; inside-ROI test of
Alg. 1 with the boxes of Eq. 1; hard voxelization with a per-voxel and a
per-frame cap; mean voxel features). Only ``tests/``, ``__graft_entry__.smoke``
and the CPU-baseline leg of ``bench.py`` may import it. It shares no code with
the CUDA library and never imports it.

The arithmetic lives in ``mmbev_oracle.c`` (plain C, built with
``-O2 -ffp-contract=off``); this module only loads it with ctypes and moves
numpy arrays in and out.

Every function here is pinned by ``tests/test_oracle_pins.py`` against facts
the paper and the mathematics fix (identity and translation transforms, the
ghost-collapse property of compensation, a brute-force polygon test,
hand-built voxels with known means, exhaustive bucketing on tiny grids and the
invariants of the cap rule).
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import sysconfig

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "mmbev_oracle.c")
_LIB = os.path.join(_HERE, "liboracle.so")

_lib = None


def build(force: bool = False) -> str:
    """Compile the oracle into ``oracle/liboracle.so`` (gcc, no contraction)."""
    if not force and os.path.exists(_LIB) and os.path.getmtime(_LIB) >= os.path.getmtime(_SRC):
        return _LIB
    cc = os.environ.get("CC", "gcc")
    tmp = _LIB + f".tmp{os.getpid()}"
    cmd = [cc, "-O2", "-ffp-contract=off", "-fno-fast-math", "-fPIC", "-shared",
           "-std=c11", "-o", tmp, _SRC, "-lm"]
    subprocess.run(cmd, check=True)
    os.replace(tmp, _LIB)
    return _LIB


def _load():
    global _lib
    if _lib is None:
        build()
        lib = ctypes.CDLL(_LIB)
        P = ctypes.c_void_p
        i32, i64, f32 = ctypes.c_int32, ctypes.c_int64, ctypes.c_float
        lib.oracle_classify.argtypes = [P, P, i32, P, P, i32, f32, P, P, P, P, P]
        lib.oracle_classify.restype = ctypes.c_int
        u64 = ctypes.c_uint64
        lib.oracle_voxelize_roi.argtypes = [P, P, i32, P, P, i32, f32, P, P,
                                            i32, i32, f32, u64, P, P, P, P]
        lib.oracle_voxelize_roi.restype = ctypes.c_int
        lib.oracle_voxelize_roi_batched.argtypes = [P, P, i32, P, P, i32, f32, P, P,
                                                    i32, i32, f32, u64, i32, P, P, P, P,
                                                    P, P]
        lib.oracle_voxelize_roi_batched.restype = ctypes.c_int
        lib.oracle_build_rois.argtypes = [P, i32, P, P, P]
        lib.oracle_build_rois.restype = ctypes.c_int
        lib.oracle_crit_thresholds.argtypes = [P, P, P]
        lib.oracle_crit_thresholds.restype = None
        lib.oracle_splitmix64.argtypes = [u64, u64]
        lib.oracle_splitmix64.restype = u64
        lib.oracle_roi_boxes.argtypes = [P, i32, f32, P]
        lib.oracle_roi_boxes.restype = None
        _lib = lib
    return _lib


def _ptr(a: np.ndarray):
    return a.ctypes.data_as(ctypes.c_void_p)


def _c(a, dtype):
    return np.ascontiguousarray(np.asarray(a, dtype=dtype))


def classify(points, sweep_offsets, sweep_tf, rois, roi_margin, voxel_size, pc_range):
    """Per point: compensated xyz (float32 [N,3]), voxel linear index (int64,
    -1 when dropped) and ROI rank (int32, -1 when dropped)."""
    lib = _load()
    points = _c(points, np.float32).reshape(-1, 5)
    so = _c(sweep_offsets, np.int64)
    tf = _c(sweep_tf, np.float32).reshape(-1, 16)
    rois = _c(rois, np.float32).reshape(-1, 5)
    vs = _c(voxel_size, np.float32)
    rg = _c(pc_range, np.float32)
    n = points.shape[0]
    xyz = np.zeros((n, 3), np.float32)
    lin = np.full(n, -1, np.int64)
    rank = np.full(n, -1, np.int32)
    rc = lib.oracle_classify(_ptr(points), _ptr(so), len(so) - 1, _ptr(tf), _ptr(rois),
                             rois.shape[0], float(roi_margin), _ptr(vs), _ptr(rg),
                             _ptr(xyz), _ptr(lin), _ptr(rank))
    if rc != 0:
        raise ValueError(f"oracle_classify failed with status {rc}")
    return xyz, lin, rank


def roi_boxes(rois, roi_margin):
    """The Eq. 1 box form of each ROI the inside test uses: float32 [R, 4] =
    (cos(yaw), sin(yaw)) from libm in double rounded to fp32, and the
    half-extents 0.5*l + r, 0.5*w + r in fp32."""
    rois = _c(rois, np.float32).reshape(-1, 5)
    out = np.zeros((rois.shape[0], 4), np.float32)
    _load().oracle_roi_boxes(_ptr(rois), rois.shape[0], float(roi_margin), _ptr(out))
    return out


def splitmix64(seed, n):
    """The n-th output (n >= 1) of the SplitMix64 stream seeded with `seed`."""
    return int(_load().oracle_splitmix64(int(seed) & (2**64 - 1), int(n) & (2**64 - 1)))


def voxelize_roi(points, sweep_offsets, sweep_tf, rois, roi_margin, voxel_size,
                 pc_range, max_pts_per_voxel, max_voxels, rho_out=0.0, seed=0):
    """One frame. Returns (feats [nvox,5], coords [nvox,3] (z,y,x), counts [nvox]).
    rho_out: keep probability of points inside no ROI (Alg. 1), drawn from
    SplitMix64(seed) per frame-local point index."""
    lib = _load()
    points = _c(points, np.float32).reshape(-1, 5)
    so = _c(sweep_offsets, np.int64)
    tf = _c(sweep_tf, np.float32).reshape(-1, 16)
    rois = _c(rois, np.float32).reshape(-1, 5)
    vs = _c(voxel_size, np.float32)
    rg = _c(pc_range, np.float32)
    mv = int(max_voxels)
    feats = np.zeros((max(mv, 1), 5), np.float32)
    coords = np.zeros((max(mv, 1), 3), np.int32)
    counts = np.zeros(max(mv, 1), np.int32)
    nvox = np.zeros(1, np.int32)
    rc = lib.oracle_voxelize_roi(_ptr(points), _ptr(so), len(so) - 1, _ptr(tf), _ptr(rois),
                                 rois.shape[0], float(roi_margin), _ptr(vs), _ptr(rg),
                                 int(max_pts_per_voxel), mv, float(rho_out),
                                 int(seed) & (2**64 - 1), _ptr(feats), _ptr(coords),
                                 _ptr(counts), _ptr(nvox))
    if rc != 0:
        raise ValueError(f"oracle_voxelize_roi failed with status {rc}")
    k = int(nvox[0])
    return feats[:k].copy(), coords[:k].copy(), counts[:k].copy()


def voxelize_roi_batched(points, sweep_offsets, sweep_tf, rois, roi_margin, voxel_size,
                         pc_range, max_pts_per_voxel, max_voxels, frame_sweep_offsets,
                         frame_roi_offsets, rho_out=0.0, seed=0):
    """Independent frames in one call. Returns a list of per-frame
    (feats, coords, counts) tuples."""
    lib = _load()
    points = _c(points, np.float32).reshape(-1, 5)
    so = _c(sweep_offsets, np.int64)
    tf = _c(sweep_tf, np.float32).reshape(-1, 16)
    rois = _c(rois, np.float32).reshape(-1, 5)
    vs = _c(voxel_size, np.float32)
    rg = _c(pc_range, np.float32)
    fso = _c(frame_sweep_offsets, np.int32)
    fro = _c(frame_roi_offsets, np.int32)
    nf = len(fso) - 1
    mv = int(max_voxels)
    rows = max(nf * mv, 1)
    feats = np.zeros((rows, 5), np.float32)
    coords = np.zeros((rows, 3), np.int32)
    counts = np.zeros(rows, np.int32)
    nvox = np.zeros(max(nf, 1), np.int32)
    rc = lib.oracle_voxelize_roi_batched(
        _ptr(points), _ptr(so), len(so) - 1, _ptr(tf), _ptr(rois), rois.shape[0],
        float(roi_margin), _ptr(vs), _ptr(rg), int(max_pts_per_voxel), mv, float(rho_out),
        int(seed) & (2**64 - 1), nf,
        _ptr(fso), _ptr(fro), _ptr(feats), _ptr(coords), _ptr(counts), _ptr(nvox))
    if rc != 0:
        raise ValueError(f"oracle_voxelize_roi_batched failed with status {rc}")
    out = []
    for f in range(nf):
        k = int(nvox[f])
        r0 = f * mv
        out.append((feats[r0:r0 + k].copy(), coords[r0:r0 + k].copy(), counts[r0:r0 + k].copy()))
    return out


CRIT_FIELDS = ("v_ego", "dt", "a_brake", "d_min", "theta_max_deg", "theta_min_deg", "v_wide",
               "v_narrow", "tau_vru", "tau_motor", "r_coll")
CLS_MOTOR, CLS_VRU, CLS_STATIC = 0, 1, 2


def _crit_params(params):
    return np.asarray([float(params[k]) for k in CRIT_FIELDS], np.float32)


def build_rois(objects, params):
    """Temporal ROIs and criticality ranking of one frame (Sec. IV-C, Eq. 1,
    3-5, 8). objects: [n, 8] float32 rows (cx, cy, w, l, yaw, vx, vy, cls).
    Returns (rois [2n, 5] in rank order, flags [n]: bit 0 Geom, bit 1 Safety)."""
    lib = _load()
    obj = np.ascontiguousarray(objects, np.float32).reshape(-1, 8)
    n = obj.shape[0]
    rec = np.zeros(n, dtype=[("f", np.float32, 7), ("cls", np.int32)])
    rec["f"] = obj[:, :7]
    rec["cls"] = obj[:, 7].astype(np.int32)
    q = _crit_params(params)
    rois = np.zeros((max(2 * n, 1), 5), np.float32)
    flags = np.zeros(max(n, 1), np.int32)
    rc = lib.oracle_build_rois(rec.ctypes.data_as(ctypes.c_void_p), n, _ptr(q), _ptr(rois),
                               _ptr(flags))
    if rc != 0:
        raise ValueError(f"oracle_build_rois failed with status {rc}")
    return rois[:2 * n].copy(), flags[:n].copy()


def crit_thresholds(params):
    """(dmax, tan(theta)) of Eq. 4 and the cone, as fp32."""
    lib = _load()
    q = _crit_params(params)
    d = np.zeros(1, np.float32)
    t = np.zeros(1, np.float32)
    lib.oracle_crit_thresholds(_ptr(q), _ptr(d), _ptr(t))
    return float(d[0]), float(t[0])


def voxel_components(frames, dims):
    """Connected components of each frame's kept voxels under 26-connectivity
    (voxels sharing a face, an edge or a corner): the voxel-grid proposer of
    the paper's robot deployment (Sec. VI-F), written out with a dict and
    union-find.
    Each voxel's label is the smallest output row (within its frame) of its
    component. Returns per frame (labels [n], components [k, 8] rows of
    (label, size, zmin, ymin, xmin, zmax, ymax, xmax) sorted by label)."""
    nx, ny, nz = (int(d) for d in dims)
    out = []
    for feats, coords, _ in frames:
        n = len(coords)
        at = {tuple(int(c) for c in coords[v]): v for v in range(n)}
        parent = list(range(n))

        def find(x):
            while parent[x] != x:
                parent[x] = parent[parent[x]]
                x = parent[x]
            return x

        for v in range(n):
            z, y, x = (int(c) for c in coords[v])
            for dz in (-1, 0, 1):
                for dy in (-1, 0, 1):
                    for dx in (-1, 0, 1):
                        u = at.get((z + dz, y + dy, x + dx))
                        if u is None or u == v:
                            continue
                        a, b = find(v), find(u)
                        if a != b:
                            parent[max(a, b)] = min(a, b)
        labels = np.array([find(v) for v in range(n)], np.int32)
        comps = {}
        for v in range(n):
            z, y, x = (int(c) for c in coords[v])
            r = comps.setdefault(int(labels[v]), [int(labels[v]), 0, z, y, x, z, y, x])
            r[1] += 1
            r[2], r[3], r[4] = min(r[2], z), min(r[3], y), min(r[4], x)
            r[5], r[6], r[7] = max(r[5], z), max(r[6], y), max(r[7], x)
        comp = np.array([comps[k] for k in sorted(comps)], np.int32).reshape(-1, 8)
        out.append((labels, comp))
    return out


def scatter_bev(frames, dims):
    """ScatterToBEV (Alg. 1, last step), written out: a zero canvas
    [F, nz*5, ny, nx] and, for every kept voxel (cz, cy, cx) of frame f, its
    feature c at channel cz*5 + c of cell (cy, cx). `frames` is the list of
    per-frame (feats, coords, counts) a voxelize call returns."""
    nx, ny, nz = (int(d) for d in dims)
    canvas = np.zeros((len(frames), nz * 5, ny, nx), np.float32)
    for f, (feats, coords, _) in enumerate(frames):
        for v in range(len(coords)):
            cz, cy, cx = (int(c) for c in coords[v])
            for c in range(5):
                canvas[f, cz * 5 + c, cy, cx] = feats[v, c]
    return canvas


def grid_dims(voxel_size, pc_range):
    """(nx, ny, nz) = round-half-away((max - min) / size) in double, as the
    oracle's llround does for these positive extents."""
    vs = np.asarray(voxel_size, np.float32).astype(np.float64)
    rg = np.asarray(pc_range, np.float32).astype(np.float64)
    return tuple(int(np.floor((rg[a + 3] - rg[a]) / vs[a] + 0.5)) for a in range(3))
