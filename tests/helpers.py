"""Shared helpers for the parity tests: run the CUDA path through the C ABI
and the oracle on the same seeded workload, and compare."""
from __future__ import annotations

import numpy as np

RTOL, ATOL = 1e-5, 1e-6   # feature tolerance; integers compare exactly


def to_dev(w, dev, rois=None):
    import torch
    pts = torch.from_numpy(np.ascontiguousarray(w.points)).to(dev)
    tf = torch.from_numpy(np.ascontiguousarray(w.sweep_tf)).to(dev)
    r = w.rois if rois is None else rois
    rois_t = torch.from_numpy(np.ascontiguousarray(r, np.float32).reshape(-1, 5)).to(dev)
    return pts, tf, rois_t


def run_gpu(mmbev, w, dev, K=None, maxv=None, inject_status=0, workspace=None,
            stream=None, rho_out=0.0, seed=0):
    """Batched C-ABI call on w; returns (per-frame list of (feats, coords,
    counts), device status, workspace)."""
    import torch
    K = w.max_pts_per_voxel if K is None else K
    maxv = w.max_voxels if maxv is None else maxv
    pts, tf, rois = to_dev(w, dev)
    nf = w.num_frames
    rmax = int(np.max(np.diff(w.frame_roi_offsets))) if nf else 0
    if workspace is None:
        workspace = mmbev.new_workspace(max(w.num_points, 1), rmax, maxv, nf, w.voxel_size,
                                        w.pc_range, dev)
    out = mmbev.voxelize_roi_batched(pts, w.sweep_offsets, tf, rois, w.roi_margin, w.voxel_size,
                                     w.pc_range, K, maxv, w.frame_sweep_offsets,
                                     w.frame_roi_offsets, workspace=workspace,
                                     inject_status=inject_status, stream=stream,
                                     rho_out=rho_out, seed=seed)
    torch.cuda.synchronize(dev)
    status = mmbev.get_status(workspace)
    nvox = out.nvox.cpu().numpy()
    frames = [out.frame(f, maxv, nvox[f]) for f in range(nf)]
    return frames, status, workspace


def run_oracle(oracle, w, K=None, maxv=None, rho_out=0.0, seed=0):
    K = w.max_pts_per_voxel if K is None else K
    maxv = w.max_voxels if maxv is None else maxv
    return oracle.voxelize_roi_batched(w.points, w.sweep_offsets, w.sweep_tf, w.rois, w.roi_margin,
                                       w.voxel_size, w.pc_range, K, maxv, w.frame_sweep_offsets,
                                       w.frame_roi_offsets, rho_out=rho_out, seed=seed)


def assert_frames_equal(got, want, label=""):
    """Coordinates, counts and order bit-exact; features within RTOL/ATOL.
    Returns the fraction of feature values that are bit-identical."""
    assert len(got) == len(want), label
    same = total = 0
    for f, ((gf, gc, gn), (wf, wc, wn)) in enumerate(zip(got, want)):
        assert gc.shape == wc.shape, f"{label} frame {f}: nvox {gc.shape[0]} != {wc.shape[0]}"
        assert np.array_equal(gc, wc), f"{label} frame {f}: coords differ"
        assert np.array_equal(gn, wn), f"{label} frame {f}: counts differ"
        np.testing.assert_allclose(gf, wf, rtol=RTOL, atol=ATOL, err_msg=f"{label} frame {f}")
        same += int(np.sum(gf.view(np.uint32) == wf.view(np.uint32)))
        total += gf.size
    return same / total if total else 1.0
