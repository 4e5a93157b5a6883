"""ROI-aware multi-sweep LiDAR voxelization for GB300 (sm_103a).

Python binding of ``libmmbev.so``, the C-ABI library declared in
``include/mmbev.h``. The binding only marshals arguments: device buffers come
from PyTorch tensors (``data_ptr``), host offsets from numpy arrays, and the
stream from ``torch.cuda.current_stream()``. Every step of the path
(motion compensation, Eq. 6-7; inside-ROI test, Alg. 1 with the boxes of
Eq. 1; grouping by voxel; cap and canonical order; mean features) runs in
the library's CUDA kernels. There is no CPU fallback: if the library is
missing, ``load()`` raises.
"""
from __future__ import annotations

import ctypes
import os
from dataclasses import dataclass

import numpy as np
import torch

_PKG = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_PKG, "libmmbev.so")

NUM_STAGES = 6
DEV_TABLE_FULL = 0x1
DEV_WAIT_TIMEOUT = 0x2
DEV_BOUNDS = 0x4
STATUS_NAMES = {0: "ok", -1: "EINVAL", -2: "ECUDA", -3: "EWORKSPACE"}

_lib = None


class MMBEVError(RuntimeError):
    """A library call returned a negative status."""


class _ExecOpts(ctypes.Structure):
    _fields_ = [("stage_events", ctypes.c_void_p), ("inject_status", ctypes.c_uint32),
                ("rho_out", ctypes.c_float), ("seed", ctypes.c_uint64)]


def load():
    """Load libmmbev.so (built by ``build()``); raises if it is absent."""
    global _lib
    if _lib is not None:
        return _lib
    if not os.path.exists(LIB_PATH):
        raise ImportError(f"{LIB_PATH} is missing: run paper_2608_15437_gb300.build() first")
    lib = ctypes.CDLL(LIB_PATH)
    P, i32, i64, f32, sz = (ctypes.c_void_p, ctypes.c_int32, ctypes.c_int64, ctypes.c_float,
                            ctypes.c_size_t)
    lib.mmbev_workspace_size.argtypes = [i64, i32, i32, i32, P, P]
    lib.mmbev_workspace_size.restype = sz
    vox = [P, P, i32, P, P, i32, f32, P, P, i32, i32]
    lib.mmbev_voxelize_roi.argtypes = vox + [P, P, P, P, P, sz, P]
    lib.mmbev_voxelize_roi.restype = ctypes.c_int
    batched = vox + [i32, P, P, P, P, P, P, P, sz, P]
    lib.mmbev_voxelize_roi_batched.argtypes = batched
    lib.mmbev_voxelize_roi_batched.restype = ctypes.c_int
    lib.mmbev_pack_size.argtypes = [i32, i32]
    lib.mmbev_pack_size.restype = sz
    lib.mmbev_pack_voxels.argtypes = [P, P, P, P, i32, i32, P, sz, P]
    lib.mmbev_pack_voxels.restype = ctypes.c_int
    lib.mmbev_components_table_size.argtypes = [i32, i32]
    lib.mmbev_components_table_size.restype = sz
    lib.mmbev_voxel_components.argtypes = [P, P, i32, i32, P, P, ctypes.c_size_t, P, P, P, P, P]
    lib.mmbev_voxel_components.restype = ctypes.c_int
    lib.mmbev_build_rois.argtypes = [P, P, i32, P, P, P, P]
    lib.mmbev_build_rois.restype = ctypes.c_int
    lib.mmbev_scatter_bev.argtypes = [P, P, P, i32, i32, P, P, ctypes.c_size_t, P]
    lib.mmbev_scatter_bev_update.argtypes = [P, P, P, P, P, i32, i32, P, P, ctypes.c_size_t, P]
    lib.mmbev_scatter_bev_update.restype = ctypes.c_int
    lib.mmbev_scatter_bev.restype = ctypes.c_int
    lib.mmbev_voxelize_roi_batched_ex.argtypes = batched + [ctypes.POINTER(_ExecOpts)]
    lib.mmbev_voxelize_roi_batched_ex.restype = ctypes.c_int
    lib.mmbev_voxelize_roi_batched_host.argtypes = (
        [P, P, i32, P, P, i32, f32, P, P, i32, i32, i32, P, P, P, P, P, P, P, P, P, P, sz,
         P, sz, i32, P, P, ctypes.POINTER(_ExecOpts)])
    lib.mmbev_voxelize_roi_batched_host.restype = ctypes.c_int
    lib.mmbev_classify_points.argtypes = [P, P, i32, P, P, i32, f32, P, P, i32, P, P,
                                          P, P, P, P, sz, P]
    lib.mmbev_classify_points.restype = ctypes.c_int
    lib.mmbev_voxelize_roi_noalloc.argtypes = vox + [P, P, P, P, P, P]
    lib.mmbev_voxelize_roi_noalloc.restype = ctypes.c_int
    lib.mmbev_prep_rois.argtypes = [P, i32, f32, P, P]
    lib.mmbev_prep_rois.restype = ctypes.c_int
    lib.mmbev_get_status.argtypes = [P, sz, ctypes.POINTER(ctypes.c_uint32), P]
    lib.mmbev_get_status.restype = ctypes.c_int
    lib.mmbev_stage_name.argtypes = [i32]
    lib.mmbev_stage_name.restype = ctypes.c_char_p
    lib.mmbev_version.argtypes = []
    lib.mmbev_version.restype = ctypes.c_char_p
    _lib = lib
    return lib


def build(force: bool = False, verbose: bool = False) -> str:
    """Compile libmmbev.so for sm_103a in-tree."""
    from . import _build
    return _build.build(force=force, verbose=verbose)


def stage_names():
    lib = load()
    return [lib.mmbev_stage_name(i).decode() for i in range(NUM_STAGES)]


def _check(rc: int, what: str):
    if rc != 0:
        raise MMBEVError(f"{what} failed: {STATUS_NAMES.get(rc, rc)}")


def _host(a, dtype) -> np.ndarray:
    if isinstance(a, torch.Tensor):
        a = a.detach().cpu().numpy()
    return np.ascontiguousarray(np.asarray(a, dtype=dtype))


def _hptr(a: np.ndarray):
    return a.ctypes.data_as(ctypes.c_void_p)


def _dptr(t: torch.Tensor | None, dtype=None, name="tensor"):
    if t is None:
        return None
    if not t.is_cuda:
        raise ValueError(f"{name} must be a CUDA tensor")
    if dtype is not None and t.dtype != dtype:
        raise ValueError(f"{name} must be {dtype}, got {t.dtype}")
    if not t.is_contiguous():
        raise ValueError(f"{name} must be contiguous")
    return ctypes.c_void_p(t.data_ptr())


def _stream(stream):
    s = stream if stream is not None else torch.cuda.current_stream()
    return ctypes.c_void_p(s.cuda_stream)


def workspace_size(max_points, max_rois_per_frame, max_voxels, num_frames, voxel_size,
                   pc_range) -> int:
    vs = _host(voxel_size, np.float32)
    rg = _host(pc_range, np.float32)
    n = load().mmbev_workspace_size(int(max_points), int(max_rois_per_frame), int(max_voxels),
                                    int(num_frames), _hptr(vs), _hptr(rg))
    if n == 0:
        raise ValueError("invalid workspace size arguments")
    return int(n)


def new_workspace(max_points, max_rois_per_frame, max_voxels, num_frames, voxel_size, pc_range,
                  device="cuda") -> torch.Tensor:
    n = workspace_size(max_points, max_rois_per_frame, max_voxels, num_frames, voxel_size, pc_range)
    return torch.empty(n, dtype=torch.uint8, device=device)


def get_status(workspace: torch.Tensor, stream=None) -> int:
    """Device status bits of the last call on this workspace (synchronizes)."""
    v = ctypes.c_uint32(0)
    _check(load().mmbev_get_status(_dptr(workspace, torch.uint8, "workspace"), workspace.numel(),
                                   ctypes.byref(v), _stream(stream)), "mmbev_get_status")
    return int(v.value)


@dataclass
class Outputs:
    """Device outputs of one call; frame f's rows start at f * max_voxels."""
    feats: torch.Tensor    # float32 [F * max_voxels, 5]
    coords: torch.Tensor   # int32 [F * max_voxels, 3] (z, y, x)
    counts: torch.Tensor   # int32 [F * max_voxels]
    nvox: torch.Tensor     # int32 [F]

    @staticmethod
    def empty(num_frames: int, max_voxels: int, device="cuda") -> "Outputs":
        rows = max(num_frames * max_voxels, 1)
        return Outputs(torch.empty((rows, 5), dtype=torch.float32, device=device),
                       torch.empty((rows, 3), dtype=torch.int32, device=device),
                       torch.empty(rows, dtype=torch.int32, device=device),
                       torch.zeros(max(num_frames, 1), dtype=torch.int32, device=device))

    def frame(self, f: int, max_voxels: int, nvox: int | None = None):
        """Frame f's kept rows as host numpy arrays (feats, coords, counts)."""
        n = int(self.nvox[f].item()) if nvox is None else int(nvox)
        r0 = f * max_voxels
        return (self.feats[r0:r0 + n].cpu().numpy(), self.coords[r0:r0 + n].cpu().numpy(),
                self.counts[r0:r0 + n].cpu().numpy())


def voxelize_roi_batched(points: torch.Tensor, sweep_offsets, sweep_tf: torch.Tensor,
                         rois: torch.Tensor, roi_margin: float, voxel_size, pc_range,
                         max_pts_per_voxel: int, max_voxels: int, frame_sweep_offsets,
                         frame_roi_offsets, *, workspace: torch.Tensor,
                         out: Outputs | None = None, stream=None, stage_events=None,
                         inject_status: int = 0, rho_out: float = 0.0,
                         seed: int = 0) -> Outputs:
    """Voxelize F independent frames in one call (``mmbev_voxelize_roi_batched``).

    points [N,5] float32, sweep_tf [S,16] float32 and rois [R,5] float32 live
    on the device; sweep_offsets [S+1], frame_sweep_offsets [F+1] and
    frame_roi_offsets [F+1] are host arrays. ``stage_events``, a list of
    NUM_STAGES + 1 ``torch.cuda.Event(enable_timing=True)`` already recorded
    once, brackets each kernel of the call. ``rho_out`` keeps points inside
    no ROI with that probability (SplitMix64 draws keyed by ``seed`` and the
    point's index within its frame). ``inject_status`` is a test hook: status
    bits the call reports as if a device-side failure had set them.
    """
    lib = load()
    so = _host(sweep_offsets, np.int64)
    fso = _host(frame_sweep_offsets, np.int32)
    fro = _host(frame_roi_offsets, np.int32)
    vs = _host(voxel_size, np.float32)
    rg = _host(pc_range, np.float32)
    nf = len(fso) - 1
    if out is None:
        out = Outputs.empty(nf, int(max_voxels), device=points.device)
    args = [_dptr(points, torch.float32, "points"), _hptr(so), len(so) - 1,
            _dptr(sweep_tf, torch.float32, "sweep_tf"), _dptr(rois, torch.float32, "rois"),
            rois.shape[0] if rois.dim() > 1 else rois.numel() // 5, float(roi_margin), _hptr(vs),
            _hptr(rg), int(max_pts_per_voxel), int(max_voxels), nf, _hptr(fso), _hptr(fro),
            _dptr(out.feats), _dptr(out.coords), _dptr(out.counts), _dptr(out.nvox),
            _dptr(workspace, torch.uint8, "workspace"), workspace.numel(), _stream(stream)]
    if stage_events is None and not inject_status and not rho_out:
        rc = lib.mmbev_voxelize_roi_batched(*args)
    else:
        opts = _ExecOpts(None, int(inject_status), float(rho_out), int(seed) & (2**64 - 1))
        if stage_events is not None:
            assert len(stage_events) == NUM_STAGES + 1
            arr = (ctypes.c_void_p * len(stage_events))(*[e.cuda_event for e in stage_events])
            opts.stage_events = ctypes.cast(arr, ctypes.c_void_p)
        rc = lib.mmbev_voxelize_roi_batched_ex(*args, ctypes.byref(opts))
    _check(rc, "mmbev_voxelize_roi_batched")
    return out


def voxelize_roi(points: torch.Tensor, sweep_offsets, sweep_tf: torch.Tensor, rois: torch.Tensor,
                 roi_margin: float, voxel_size, pc_range, max_pts_per_voxel: int,
                 max_voxels: int, *, workspace: torch.Tensor,
                 out: Outputs | None = None, stream=None) -> Outputs:
    """One frame (``mmbev_voxelize_roi``); out.nvox holds one entry."""
    lib = load()
    so = _host(sweep_offsets, np.int64)
    vs = _host(voxel_size, np.float32)
    rg = _host(pc_range, np.float32)
    if out is None:
        out = Outputs.empty(1, int(max_voxels), device=points.device)
    nr = rois.shape[0] if rois.dim() > 1 else rois.numel() // 5
    rc = lib.mmbev_voxelize_roi(
        _dptr(points, torch.float32, "points"), _hptr(so), len(so) - 1,
        _dptr(sweep_tf, torch.float32, "sweep_tf"), _dptr(rois, torch.float32, "rois"), nr,
        float(roi_margin), _hptr(vs), _hptr(rg), int(max_pts_per_voxel), int(max_voxels),
        _dptr(out.feats), _dptr(out.coords), _dptr(out.counts), _dptr(out.nvox),
        _dptr(workspace, torch.uint8, "workspace"), workspace.numel(), _stream(stream))
    _check(rc, "mmbev_voxelize_roi")
    return out


def voxelize_roi_noalloc(points: torch.Tensor, sweep_offsets, sweep_tf: torch.Tensor,
                         rois: torch.Tensor, roi_margin: float, voxel_size, pc_range,
                         max_pts_per_voxel: int, max_voxels: int, *, out: Outputs,
                         status: torch.Tensor | None = None, stream=None) -> Outputs:
    """One frame without a workspace (``mmbev_voxelize_roi_noalloc``),
    for callers that cannot allocate device memory: the library's own
    file-scope device array serves as scratch. ``out`` (and ``status``, a
    1-element uint32/int32 device tensor) must be allocated by the caller."""
    lib = load()
    so = _host(sweep_offsets, np.int64)
    vs = _host(voxel_size, np.float32)
    rg = _host(pc_range, np.float32)
    nr = rois.shape[0] if rois.dim() > 1 else rois.numel() // 5
    rc = lib.mmbev_voxelize_roi_noalloc(
        _dptr(points, torch.float32, "points"), _hptr(so), len(so) - 1,
        _dptr(sweep_tf, torch.float32, "sweep_tf"), _dptr(rois, torch.float32, "rois"), nr,
        float(roi_margin), _hptr(vs), _hptr(rg), int(max_pts_per_voxel), int(max_voxels),
        _dptr(out.feats), _dptr(out.coords), _dptr(out.counts), _dptr(out.nvox),
        _dptr(status), _stream(stream))
    _check(rc, "mmbev_voxelize_roi_noalloc")
    return out


def classify_points(points: torch.Tensor, sweep_offsets, sweep_tf: torch.Tensor,
                    rois: torch.Tensor, roi_margin: float, voxel_size, pc_range,
                    frame_sweep_offsets, frame_roi_offsets, *, workspace: torch.Tensor,
                    stream=None):
    """Steps S1-S2 per point: (xyz [N,3] f32, lin [N] i64, rank [N] i32) on the device."""
    lib = load()
    so = _host(sweep_offsets, np.int64)
    fso = _host(frame_sweep_offsets, np.int32)
    fro = _host(frame_roi_offsets, np.int32)
    vs = _host(voxel_size, np.float32)
    rg = _host(pc_range, np.float32)
    n = int(so[-1])
    dev = points.device
    xyz = torch.empty((max(n, 1), 3), dtype=torch.float32, device=dev)
    lin = torch.empty(max(n, 1), dtype=torch.int64, device=dev)
    rank = torch.empty(max(n, 1), dtype=torch.int32, device=dev)
    nr = rois.shape[0] if rois.dim() > 1 else rois.numel() // 5
    rc = lib.mmbev_classify_points(
        _dptr(points, torch.float32, "points"), _hptr(so), len(so) - 1,
        _dptr(sweep_tf, torch.float32, "sweep_tf"), _dptr(rois, torch.float32, "rois"), nr,
        float(roi_margin), _hptr(vs), _hptr(rg), len(fso) - 1, _hptr(fso), _hptr(fro),
        _dptr(xyz), _dptr(lin), _dptr(rank), _dptr(workspace, torch.uint8, "workspace"),
        workspace.numel(), _stream(stream))
    _check(rc, "mmbev_classify_points")
    return xyz[:n], lin[:n], rank[:n]


def prep_rois(rois: torch.Tensor, roi_margin: float, stream=None) -> torch.Tensor:
    """The prepared boxes the inside test uses (``mmbev_prep_rois``): float32
    [R, 6] = (cx, cy, cos(yaw), sin(yaw), hl, hw) as the device computes them."""
    lib = load()
    nr = rois.shape[0] if rois.dim() > 1 else rois.numel() // 5
    out = torch.empty((max(nr, 1), 6), dtype=torch.float32, device=rois.device)
    rc = lib.mmbev_prep_rois(_dptr(rois, torch.float32, "rois"), nr, float(roi_margin),
                             _dptr(out), _stream(stream))
    _check(rc, "mmbev_prep_rois")
    return out[:nr]


CRIT_FIELDS = ("v_ego", "dt", "a_brake", "d_min", "theta_max_deg", "theta_min_deg", "v_wide",
               "v_narrow", "tau_vru", "tau_motor", "r_coll")
CLS_MOTOR, CLS_VRU, CLS_STATIC = 0, 1, 2


def pack_bytes(num_frames: int, max_voxels: int) -> int:
    """Bytes ``pack_voxels`` may write for this batch shape."""
    return int(load().mmbev_pack_size(int(num_frames), int(max_voxels)))


def pack_voxels(out: "Outputs", max_voxels: int, dst: torch.Tensor, stream=None) -> None:
    """Gather every frame's kept rows into dst (``mmbev_pack_voxels``): a
    uint8 tensor of at least ``pack_bytes`` bytes, on the device or in pinned
    host memory (the device then writes it directly). Read it back with
    ``unpack``."""
    lib = load()
    nf = out.nvox.numel()
    if dst.dtype != torch.uint8 or not dst.is_contiguous():
        raise ValueError("dst must be a contiguous uint8 tensor")
    if not dst.is_cuda and not dst.is_pinned():
        raise ValueError("dst must be on the device or in pinned host memory")
    rc = lib.mmbev_pack_voxels(_dptr(out.feats), _dptr(out.coords), _dptr(out.counts),
                               _dptr(out.nvox), nf, int(max_voxels),
                               ctypes.c_void_p(dst.data_ptr()), dst.numel(), _stream(stream))
    _check(rc, "mmbev_pack_voxels")


def unpack(dst: torch.Tensor, num_frames: int):
    """Views of a packed buffer: (off [F+1] int32, feats [T,5] fp32, coords
    [T,3] int32, counts [T] int32)."""
    words = dst.view(torch.int32)
    off = words[:num_frames + 1]
    total = int(off[-1])
    rec = words[num_frames + 1:num_frames + 1 + 9 * total].view(total, 9)
    return off, rec[:, :5].view(torch.float32), rec[:, 5:8], rec[:, 8]


def components_table_bytes(num_frames: int, max_voxels: int) -> int:
    """Bytes of all-zero table ``voxel_components`` needs (0: none, as for
    every cap up to 262,144 voxels a frame)."""
    return int(load().mmbev_components_table_size(int(num_frames), int(max_voxels)))


def voxel_components(out: "Outputs", max_voxels: int, dims, table: torch.Tensor | None = None,
                     stream=None):
    """Connected components of the kept voxels (``mmbev_voxel_components``,
    26-connectivity). table: None when ``components_table_bytes`` is 0, else
    an all-zero uint8 device buffer of at least that size. Returns (labels [F*max_voxels] int32: the frame-local root row, -1
    for unused rows; comp [F*max_voxels, 7] int32: size and box at root rows;
    ncomp [F] int32; status [1] uint32)."""
    lib = load()
    nf = out.nvox.numel()
    dev = out.coords.device
    rows = max(nf * int(max_voxels), 1)
    labels = torch.empty(rows, dtype=torch.int32, device=dev)
    comp = torch.empty((rows, 7), dtype=torch.int32, device=dev)
    ncomp = torch.empty(max(nf, 1), dtype=torch.int32, device=dev)
    status = torch.zeros(1, dtype=torch.int32, device=dev)
    d = np.asarray([int(x) for x in dims], np.int32)
    rc = lib.mmbev_voxel_components(_dptr(out.coords), _dptr(out.nvox), nf, int(max_voxels),
                                    _hptr(d), _dptr(table, torch.uint8, "table"),
                                    0 if table is None else table.numel(),
                                    _dptr(labels), _dptr(comp), _dptr(ncomp), _dptr(status),
                                    _stream(stream))
    _check(rc, "mmbev_voxel_components")
    return labels, comp, ncomp[:nf], status


def pack_objects(objects: torch.Tensor) -> torch.Tensor:
    """float32 [n, 8] rows (cx, cy, w, l, yaw, vx, vy, class) on the device ->
    the ``mmbev_object_t`` layout (the class as int32 bits in column 7)."""
    n = objects.shape[0]
    packed = torch.empty((max(n, 1), 8), dtype=torch.float32, device=objects.device)
    if n:
        packed[:n, :7] = objects[:, :7]
        packed.view(torch.int32)[:n, 7] = objects[:, 7].to(torch.int32)
    return packed[:n]


def build_rois(packed: torch.Tensor, frame_obj_offsets, params: dict, out=None, stream=None):
    """Temporal ROIs and criticality ranking (``mmbev_build_rois``).

    packed: device objects from ``pack_objects`` (class 0 motorized,
    1 vulnerable, 2 static); frame_obj_offsets: host [F+1]; params: the
    CRIT_FIELDS; out: optional (rois, flags) to fill. Returns (rois [2n, 5]
    float32 in rank order per frame, flags [n] int32, frame_roi_offsets =
    2 * offsets)."""
    lib = load()
    off = _host(frame_obj_offsets, np.int32)
    n = packed.shape[0]
    dev = packed.device
    if out is None:
        out = (torch.empty((max(2 * n, 1), 5), dtype=torch.float32, device=dev),
               torch.empty(max(n, 1), dtype=torch.int32, device=dev))
    rois, flags = out
    q = np.asarray([float(params[k]) for k in CRIT_FIELDS], np.float32)
    rc = lib.mmbev_build_rois(_dptr(packed) if n else None, _hptr(off), len(off) - 1, _hptr(q),
                              _dptr(rois), _dptr(flags), _stream(stream))
    _check(rc, "mmbev_build_rois")
    return rois[:2 * n], flags[:n], (2 * off).astype(np.int32)


def scatter_bev(out: "Outputs", max_voxels: int, dims, canvas: torch.Tensor | None = None,
                stream=None) -> torch.Tensor:
    """ScatterToBEV (``mmbev_scatter_bev``): the voxels of a voxelize call's
    outputs written into a zero-filled fp32 canvas [F, nz*5, ny, nx] (channel
    cz*5 + c of cell (cy, cx) holds feature c of voxel (cz, cy, cx))."""
    lib = load()
    nx, ny, nz = (int(d) for d in dims)
    nf = out.nvox.numel()
    if canvas is None:
        canvas = torch.empty((nf, nz * 5, ny, nx), dtype=torch.float32, device=out.feats.device)
    d = np.asarray([nx, ny, nz], np.int32)
    rc = lib.mmbev_scatter_bev(_dptr(out.feats), _dptr(out.coords), _dptr(out.nvox), nf,
                               int(max_voxels), _hptr(d), _dptr(canvas, torch.float32, "canvas"),
                               canvas.numel() * 4, _stream(stream))
    _check(rc, "mmbev_scatter_bev")
    return canvas


def scatter_bev_update(prev: "Outputs | None", out: "Outputs", max_voxels: int, dims,
                       canvas: torch.Tensor, stream=None) -> torch.Tensor:
    """ScatterToBEV into a canvas that holds exactly the scatter of ``prev``
    (``mmbev_scatter_bev_update``; None: an all-zero canvas): the cells of
    prev's voxels are zeroed, then out's written, giving the canvas
    ``scatter_bev(out)`` would. ``prev`` and ``out`` must be different
    buffers (double-buffer the outputs)."""
    lib = load()
    nx, ny, nz = (int(d) for d in dims)
    nf = out.nvox.numel()
    d = np.asarray([nx, ny, nz], np.int32)
    rc = lib.mmbev_scatter_bev_update(
        None if prev is None else _dptr(prev.coords), None if prev is None else _dptr(prev.nvox),
        _dptr(out.feats), _dptr(out.coords), _dptr(out.nvox), nf, int(max_voxels), _hptr(d),
        _dptr(canvas, torch.float32, "canvas"), canvas.numel() * 4, _stream(stream))
    _check(rc, "mmbev_scatter_bev_update")
    return canvas


class Voxelizer:
    """Owns a workspace sized for one workload shape and runs the batched
    entry point on device tensors."""

    def __init__(self, max_points, max_rois_per_frame, max_voxels, num_frames, voxel_size,
                 pc_range, max_pts_per_voxel, roi_margin, device="cuda", rho_out=0.0, seed=0):
        self.rho_out = float(rho_out)
        self.seed = int(seed)
        self.voxel_size = _host(voxel_size, np.float32)
        self.pc_range = _host(pc_range, np.float32)
        self.max_voxels = int(max_voxels)
        self.K = int(max_pts_per_voxel)
        self.margin = float(roi_margin)
        self.num_frames = int(num_frames)
        self.workspace = new_workspace(max_points, max_rois_per_frame, max_voxels, num_frames,
                                       voxel_size, pc_range, device)
        self.out = Outputs.empty(num_frames, self.max_voxels, device)

    def __call__(self, points, sweep_offsets, sweep_tf, rois, frame_sweep_offsets,
                 frame_roi_offsets, stream=None, stage_events=None) -> Outputs:
        return voxelize_roi_batched(points, sweep_offsets, sweep_tf, rois, self.margin,
                                    self.voxel_size, self.pc_range, self.K, self.max_voxels,
                                    frame_sweep_offsets, frame_roi_offsets,
                                    workspace=self.workspace, out=self.out, stream=stream,
                                    stage_events=stage_events, rho_out=self.rho_out,
                                    seed=self.seed)

    def run_host(self, h_points: torch.Tensor, sweep_offsets, h_sweep_tf: torch.Tensor,
                 h_rois: torch.Tensor, frame_sweep_offsets, frame_roi_offsets,
                 chunk_frames: int = 8, stream=None, pack_dst: torch.Tensor | None = None,
                 inject_status: int = 0) -> Outputs:
        """The batched call on pinned host inputs
        (``mmbev_voxelize_roi_batched_host``): chunks of ``chunk_frames``
        frames go up on a side stream while earlier chunks are voxelized.
        With ``pack_dst`` (a uint8 tensor of ``pack_bytes``, on the device or
        pinned), each chunk's kept rows are packed there as it completes.
        Device staging is allocated on first use and kept: two sets, used in
        turn, so that a call's uploads can run while the previous call still
        computes (they wait only for the call before that one to have
        finished reading the set they overwrite). ``inject_status`` is the
        test hook of ``voxelize_roi_batched``, applied to the first chunk."""
        if pack_dst is not None and (pack_dst.dtype != torch.uint8 or not pack_dst.is_contiguous()
                                     or not (pack_dst.is_cuda or pack_dst.is_pinned())):
            raise ValueError("pack_dst must be a contiguous uint8 device or pinned tensor")
        lib = load()
        so = _host(sweep_offsets, np.int64)
        fso = _host(frame_sweep_offsets, np.int32)
        fro = _host(frame_roi_offsets, np.int32)
        for name, t in (("h_points", h_points), ("h_sweep_tf", h_sweep_tf), ("h_rois", h_rois)):
            if t.is_cuda or t.dtype != torch.float32 or not t.is_contiguous():
                raise ValueError(f"{name} must be a contiguous float32 host tensor")
        dev = self.out.nvox.device
        need = (h_points.shape, h_sweep_tf.shape, h_rois.shape)
        if getattr(self, "_staging_shape", None) != need:
            self._staging = [tuple(torch.empty(sh, dtype=torch.float32, device=dev) for sh in need)
                             for _ in range(2)]
            self._staging_read = [None, None]   # event: the last call using the set is done
            self._staging_next = 0
            self._staging_shape = need
            self._copy_stream = torch.cuda.Stream(device=dev)
        k = self._staging_next
        self._staging_next = 1 - k
        d_pts, d_tf, d_rois = self._staging[k]
        st = stream if stream is not None else torch.cuda.current_stream(dev)
        # this call's copies overwrite set k: they start once the call that
        # last read it has finished (on first use, after the earlier work on
        # `st`)
        if self._staging_read[k] is None:
            self._copy_stream.wait_stream(st)
        else:
            self._copy_stream.wait_event(self._staging_read[k])
        opts = _ExecOpts(None, int(inject_status), float(self.rho_out),
                         int(self.seed) & (2**64 - 1))
        nr = h_rois.shape[0] if h_rois.dim() > 1 else h_rois.numel() // 5
        rc = lib.mmbev_voxelize_roi_batched_host(
            ctypes.c_void_p(h_points.data_ptr()), _hptr(so), len(so) - 1,
            ctypes.c_void_p(h_sweep_tf.data_ptr()), ctypes.c_void_p(h_rois.data_ptr()), nr,
            self.margin, _hptr(self.voxel_size), _hptr(self.pc_range), self.K, self.max_voxels,
            len(fso) - 1, _hptr(fso), _hptr(fro), _dptr(d_pts), _dptr(d_tf), _dptr(d_rois),
            _dptr(self.out.feats), _dptr(self.out.coords), _dptr(self.out.counts),
            _dptr(self.out.nvox), _dptr(self.workspace), self.workspace.numel(),
            None if pack_dst is None else ctypes.c_void_p(pack_dst.data_ptr()),
            0 if pack_dst is None else pack_dst.numel(), int(chunk_frames), _stream(st),
            _stream(self._copy_stream),
            ctypes.byref(opts))
        _check(rc, "mmbev_voxelize_roi_batched_host")
        done = torch.cuda.Event()
        done.record(st)
        self._staging_read[k] = done
        return self.out

    def status(self) -> int:
        return get_status(self.workspace)
