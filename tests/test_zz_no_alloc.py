"""The no-allocation entry point against the workspace entry point.

mmbev_voxelize_roi_noalloc serves callers that cannot allocate device memory
(for example a real-time process that forbids cudaMalloc after start-up, or a
host that lends the library only its input and output buffers): its
workspace is the library's own file-scope device array. Two calls in a
row, on frames of different shapes, must give what mmbev_voxelize_roi gives
with caller-owned buffers, so the second call also shows that the shared
array's leftovers from the first do not leak into it. This file is collected
last on purpose.
"""
import numpy as np
import pytest
import torch

import synth
from helpers import assert_frames_equal, to_dev

pytestmark = pytest.mark.gpu


def _with_workspace(mmbev, w, dev):
    pts, tf, rois = to_dev(w, dev)
    ws = mmbev.new_workspace(w.num_points, w.rois.shape[0], w.max_voxels, 1, w.voxel_size,
                             w.pc_range, dev)
    out = mmbev.voxelize_roi(pts, w.sweep_offsets, tf, rois, w.roi_margin, w.voxel_size,
                             w.pc_range, w.max_pts_per_voxel, w.max_voxels, workspace=ws)
    torch.cuda.synchronize(dev)
    assert mmbev.get_status(ws) == 0
    return [out.frame(0, w.max_voxels)]


def _no_alloc(mmbev, w, dev):
    pts, tf, rois = to_dev(w, dev)
    out = mmbev.Outputs.empty(1, w.max_voxels, dev)
    status = torch.full((1,), 0x7FFFFFFF, dtype=torch.int32, device=dev)
    mmbev.voxelize_roi_noalloc(pts, w.sweep_offsets, tf, rois, w.roi_margin, w.voxel_size,
                               w.pc_range, w.max_pts_per_voxel, w.max_voxels, out=out,
                               status=status)
    torch.cuda.synchronize(dev)
    assert int(status.item()) == 0
    return [out.frame(0, w.max_voxels)]


def test_no_alloc_matches_workspace_entry_on_two_calls(mmbev_lib, cuda_dev):
    first = synth.nuscenes_frame(1)      # 347,200 points, K = 10
    second = synth.ouster_frame(2)       # 393,216 points, K = 5, another layout
    for w in (first, second):
        want = _with_workspace(mmbev_lib, w, cuda_dev)
        got = _no_alloc(mmbev_lib, w, cuda_dev)
        assert got[0][1].shape[0] > 1000
        assert_frames_equal(got, want, f"no-alloc {w.name}")


def test_no_alloc_rejects_calls_beyond_its_array(mmbev_lib, cuda_dev):
    w = synth.concat_frames([synth.nuscenes_frame(s) for s in range(1, 6)], "five")
    need = mmbev_lib.workspace_size(w.num_points, w.rois.shape[0], 1000, 1, w.voxel_size,
                                    w.pc_range)
    assert need > 96 * 2**20           # more than the array holds
    pts, tf, rois = to_dev(w, cuda_dev)
    out = mmbev_lib.Outputs.empty(1, 1000, cuda_dev)
    with pytest.raises(mmbev_lib.MMBEVError, match="EWORKSPACE"):
        mmbev_lib.voxelize_roi_noalloc(pts, w.sweep_offsets, tf, rois, w.roi_margin,
                                       w.voxel_size, w.pc_range, 10, 1000, out=out)
