"""GPU parity: the CUDA path, called through the C ABI, against the oracle on
the same seeded inputs.

Voxel coordinates, counts, the kept-point selection (first K by index) and
the voxel order are compared bit-exactly; features within 1e-5 relative /
1e-6 absolute (the bound the kernels are built to meet exactly: both sides
sum in index order with the same fp32 operations, so the measured bit-exact
fraction is reported as well). Covers all five workload shapes at full size,
the cap path, and the edge cases of the method.
"""
import numpy as np
import pytest

import synth
from helpers import assert_frames_equal, run_gpu, run_oracle, to_dev

pytestmark = pytest.mark.gpu


def _table_is_clean(table):
    return not bool(table.any().item())


# ------------------------------------------------------------------ S1 + S2 per point

@pytest.mark.parametrize("name", ["tiny", "nuscenes", "ouster", "roi_128", "roi_full"])
def test_classify_bit_exact(oracle_mod, mmbev_lib, cuda_dev, name):
    w = synth.CONFIGS[name]()
    pts, tf, rois = to_dev(w, cuda_dev)
    ws = mmbev_lib.new_workspace(w.num_points, w.rois.shape[0], 0, 1, w.voxel_size, w.pc_range,
                                 cuda_dev)
    xyz, lin, rank = mmbev_lib.classify_points(pts, w.sweep_offsets, tf, rois, w.roi_margin,
                                               w.voxel_size, w.pc_range, w.frame_sweep_offsets,
                                               w.frame_roi_offsets, workspace=ws)
    exyz, elin, erank = oracle_mod.classify(w.points, w.sweep_offsets, w.sweep_tf, w.rois,
                                            w.roi_margin, w.voxel_size, w.pc_range)
    assert np.array_equal(xyz.cpu().numpy().view(np.uint32), exyz.view(np.uint32))
    assert np.array_equal(lin.cpu().numpy(), elin)
    assert np.array_equal(rank.cpu().numpy(), erank)


def test_roi_prep_trig_matches_libm_on_a_million_yaws(oracle_mod, mmbev_lib, cuda_dev):
    """The device's fp32 cos/sin of each yaw (CUDA's double cos/sin, rounded)
    against the oracle's (libm's double cos/sin, rounded), bit for bit: the
    two agree unless a double result lies within an ulp of an fp32 rounding
    boundary, which would flip points on an ROI edge (Eq. 1; Alg. 1's inside
    test). 1,200,000 yaws uniform over eight turns, plus every multiple of
    pi/4 in that span and its three fp32 neighbours on each side."""
    import torch
    rng = np.random.default_rng(11)
    n = 1_200_000
    yaws = rng.uniform(-8 * np.pi, 8 * np.pi, n).astype(np.float32)
    k = (np.arange(-32, 33) * (np.pi / 4)).astype(np.float32)
    extra = [k]
    up, dn = k, k
    for _ in range(3):
        up = np.nextafter(up, np.float32(np.inf))
        dn = np.nextafter(dn, np.float32(-np.inf))
        extra += [up, dn]
    yaws = np.concatenate([yaws] + extra).astype(np.float32)
    rois = np.zeros((yaws.size, 5), np.float32)
    rois[:, 0] = rng.uniform(-50, 50, yaws.size)
    rois[:, 1] = rng.uniform(-50, 50, yaws.size)
    rois[:, 2] = rng.uniform(0.5, 6, yaws.size)
    rois[:, 3] = rng.uniform(0.5, 12, yaws.size)
    rois[:, 4] = yaws
    margin = 0.37
    got = mmbev_lib.prep_rois(torch.from_numpy(rois).to(cuda_dev), margin).cpu().numpy()
    want = oracle_mod.roi_boxes(rois, margin)
    assert yaws.size > 1_000_000
    assert np.array_equal(got[:, 0:2].view(np.uint32), rois[:, 0:2].view(np.uint32))
    bad = np.nonzero(np.any(got[:, 2:6].view(np.uint32) != want.view(np.uint32), axis=1))[0]
    assert bad.size == 0, f"{bad.size} of {yaws.size} ROIs differ, e.g. yaw {yaws[bad[:5]]}"


# ------------------------------------------------------------------ whole path, full sizes

@pytest.mark.parametrize("name", ["tiny", "nuscenes", "ouster", "roi_0", "roi_8", "roi_32",
                                  "roi_128", "roi_full"])
def test_voxelize_parity(oracle_mod, mmbev_lib, cuda_dev, name):
    w = synth.CONFIGS[name]()
    got, status, _ = run_gpu(mmbev_lib, w, cuda_dev)
    assert status == 0
    want = run_oracle(oracle_mod, w)
    exact = assert_frames_equal(got, want, name)
    assert exact == 1.0, f"{name}: {exact:.6f} of feature values bit-exact"


@pytest.mark.parametrize("n_rois", [33, 48, 64, 65, 96])
def test_mask_sizes_between_the_configs(oracle_mod, mmbev_lib, cuda_dev, n_rois):
    """ROI counts whose candidate masks the configs do not reach: two mask
    words per cell on the 64 x 64 grid (33-64 ROIs: 32 KB per staged frame,
    a ring of three tiles) and three words on a 36 x 36 grid (65-96 ROIs),
    over three frames, so blocks stage two frames."""
    w = synth.concat_frames([synth.roi_coverage(n_rois, scene_seed=s) for s in (1, 2, 3)],
                            f"roi{n_rois}x3")
    got, status, _ = run_gpu(mmbev_lib, w, cuda_dev)
    assert status == 0
    want = run_oracle(oracle_mod, w)
    assert assert_frames_equal(got, want, w.name) == 1.0


def test_batch32_parity(oracle_mod, mmbev_lib, cuda_dev):
    """The benchmark's workload and launch configuration: 32 frames, 11.1 M
    points, one call."""
    w = synth.streaming_batch(32)
    got, status, _ = run_gpu(mmbev_lib, w, cuda_dev)
    assert status == 0
    want = run_oracle(oracle_mod, w)
    assert assert_frames_equal(got, want, "batch32") == 1.0


_DENSE = {}


def _dense_workload(oracle_mod):
    """Four batch frames, checked (oracle side, once) to hold a voxel of more
    than 4,096 kept points: its run in the sorted keys spans more than one
    tile of a radix pass (4,096 items) and of the voxel numbering (2,048)."""
    if "w" not in _DENSE:
        w = synth.streaming_batch(4)
        big = 0
        for f in range(w.num_frames):
            fr = w.frame(f)
            _, lin, _ = oracle_mod.classify(fr.points, fr.sweep_offsets, fr.sweep_tf, fr.rois,
                                            fr.roi_margin, fr.voxel_size, fr.pc_range)
            kept = lin[lin >= 0]
            if kept.size:
                big = max(big, int(np.unique(kept, return_counts=True)[1].max()))
        _DENSE["w"], _DENSE["big"] = w, big
    assert _DENSE["big"] > 4096
    return _DENSE["w"]


@pytest.mark.parametrize("K", [1, 10, 33, 64])
def test_dense_voxels_across_tiles(oracle_mod, mmbev_lib, cuda_dev, K):
    """Runs of thousands of points (one voxel) across radix and numbering
    tiles keep their first K points by index, at every output instantiation
    that the K values select."""
    w = _dense_workload(oracle_mod)
    want = run_oracle(oracle_mod, w, K=K)
    got, status, _ = run_gpu(mmbev_lib, w, cuda_dev, K=K)
    assert status == 0
    assert assert_frames_equal(got, want, f"dense voxels, K={K}") == 1.0


@pytest.mark.parametrize("vs", [(0.05, 0.05, 0.2), (0.03, 0.03, 0.1)])
def test_lins_of_four_digits(oracle_mod, mmbev_lib, cuda_dev, vs):
    """Grids of more than 2^27 cells over the nuScenes-shaped range
    (2,160 x 2,160 x 40 and 3,600 x 3,600 x 80): lins of 28 and 30 bits take
    four 9-bit radix passes, the last on the top digit, and the sorted items
    end in the first of the two buffers again."""
    w = synth.nuscenes_frame()
    w.voxel_size = np.array(vs, np.float32)
    got, status, _ = run_gpu(mmbev_lib, w, cuda_dev)
    assert status == 0
    want = run_oracle(oracle_mod, w)
    assert assert_frames_equal(got, want, f"voxel size {vs}") == 1.0


# ------------------------------------------------------------------ cap path

@pytest.mark.parametrize("maxv", [1, 777, 5000, 13000])
def test_cap_parity(oracle_mod, mmbev_lib, cuda_dev, maxv):
    w = synth.nuscenes_frame(1)
    got, status, _ = run_gpu(mmbev_lib, w, cuda_dev, maxv=maxv)
    want = run_oracle(oracle_mod, w, maxv=maxv)
    assert status == 0
    assert got[0][1].shape[0] == maxv
    assert_frames_equal(got, want, f"cap {maxv}")


def test_cap_full_coverage_and_mixed_frames(oracle_mod, mmbev_lib, cuda_dev):
    # frames with and without the cap in one call; one frame has no ROIs
    frames = [synth.roi_coverage("full"), synth.tiny(3), synth.roi_coverage(128),
              synth.roi_coverage(0)]
    for f in frames:
        f.max_voxels = 40000
        f.max_pts_per_voxel = 10
    b = synth.concat_frames(frames, "mixed")
    got, status, _ = run_gpu(mmbev_lib, b, cuda_dev)
    want = run_oracle(oracle_mod, b)
    assert status == 0
    assert_frames_equal(got, want, "mixed")
    assert [g[1].shape[0] for g in got][0] == 40000


def test_max_voxels_zero(oracle_mod, mmbev_lib, cuda_dev):
    w = synth.tiny(0)
    got, status, _ = run_gpu(mmbev_lib, w, cuda_dev, maxv=0)
    assert status == 0 and got[0][1].shape[0] == 0


# ------------------------------------------------------------------ per-voxel cap K

@pytest.mark.parametrize("K", [1, 3, 12, 20, 33, 64])   # every k_emit instantiation
def test_points_per_voxel(oracle_mod, mmbev_lib, cuda_dev, K):
    w = synth.nuscenes_frame(1)
    got, status, _ = run_gpu(mmbev_lib, w, cuda_dev, K=K)
    want = run_oracle(oracle_mod, w, K=K)
    assert status == 0
    assert_frames_equal(got, want, f"K={K}")


# ------------------------------------------------------------------ edge cases

def _custom(points, offsets, tfs, rois, margin=0.5, vs=(0.2, 0.2, 8.0),
            rg=(-51.2, -51.2, -5.0, 51.2, 51.2, 3.0), K=10, maxv=1000, fso=None, fro=None):
    return synth.Workload(
        name="custom", points=np.asarray(points, np.float32).reshape(-1, 5),
        sweep_offsets=np.asarray(offsets, np.int64), sweep_tf=np.asarray(tfs, np.float32).reshape(-1, 16),
        rois=np.asarray(rois, np.float32).reshape(-1, 5), roi_margin=margin,
        voxel_size=np.asarray(vs, np.float32), pc_range=np.asarray(rg, np.float32),
        max_pts_per_voxel=K, max_voxels=maxv,
        frame_sweep_offsets=None if fso is None else np.asarray(fso, np.int32),
        frame_roi_offsets=None if fro is None else np.asarray(fro, np.int32))


EYE = np.eye(4, dtype=np.float32).reshape(16)
FULL = [[0.0, 0.0, 1000.0, 1000.0, 0.0]]


def test_empty_input(oracle_mod, mmbev_lib, cuda_dev):
    w = _custom(np.zeros((0, 5)), [0, 0], [EYE], FULL)
    got, status, _ = run_gpu(mmbev_lib, w, cuda_dev)
    assert status == 0 and got[0][1].shape[0] == 0


def test_no_rois(oracle_mod, mmbev_lib, cuda_dev):
    w = synth.tiny(0).with_rois(np.zeros((0, 5), np.float32))
    got, status, _ = run_gpu(mmbev_lib, w, cuda_dev)
    assert status == 0 and got[0][1].shape[0] == 0


def test_ragged_tiles_and_empty_sweeps(oracle_mod, mmbev_lib, cuda_dev):
    # 5 sweeps, two of them empty, N = 6,151 (not a multiple of 4 or 2048);
    # each sweep shifted, so the sweep lookup matters.
    rng = np.random.default_rng(21)
    sizes = [2047, 0, 2050, 0, 2054]
    offs = np.concatenate([[0], np.cumsum(sizes)])
    n = offs[-1]
    pts = np.zeros((n, 5), np.float32)
    pts[:, 0] = rng.uniform(-20, 20, n)
    pts[:, 1] = rng.uniform(-20, 20, n)
    pts[:, 2] = rng.uniform(-4, 2, n)
    pts[:, 3] = rng.uniform(0, 1, n)
    pts[:, 4] = np.repeat(np.arange(5) * 0.05, sizes)
    tfs = []
    for s in range(5):
        t = np.eye(4, dtype=np.float32)
        t[0, 3], t[1, 3] = 0.37 * s, -0.21 * s
        tfs.append(t.reshape(16))
    rois = [[0, 0, 8, 12, 0.4], [5, 5, 3, 3, 1.0], [-10, 3, 6, 2, 2.0]]
    w = _custom(pts, offs, tfs, rois, vs=(0.1, 0.1, 0.2), K=4, maxv=100000)
    got, status, _ = run_gpu(mmbev_lib, w, cuda_dev)
    assert status == 0
    assert_frames_equal(got, run_oracle(oracle_mod, w), "ragged")
    assert got[0][1].shape[0] > 100


def test_many_sweeps_per_tile(oracle_mod, mmbev_lib, cuda_dev):
    # 300 sweeps of 7 points: a 2048-point tile spans more sweeps than the
    # kernel stages in shared memory, taking the per-point lookup.
    rng = np.random.default_rng(22)
    S, m = 300, 7
    n = S * m
    pts = np.zeros((n, 5), np.float32)
    pts[:, :2] = rng.uniform(-10, 10, (n, 2))
    pts[:, 2] = rng.uniform(-2, 2, n)
    pts[:, 3] = rng.uniform(0, 1, n)
    tfs = []
    for s in range(S):
        t = np.eye(4, dtype=np.float32)
        t[0, 3] = 0.01 * s
        tfs.append(t.reshape(16))
    w = _custom(pts, np.arange(S + 1) * m, tfs, FULL, vs=(0.5, 0.5, 0.5), K=3, maxv=100000)
    got, status, _ = run_gpu(mmbev_lib, w, cuda_dev)
    assert status == 0
    assert_frames_equal(got, run_oracle(oracle_mod, w), "many sweeps")


def test_non_finite_and_boundary_points(oracle_mod, mmbev_lib, cuda_dev):
    up = lambda v: float(np.nextafter(np.float32(v), np.float32(np.inf)))
    below = lambda v: float(np.nextafter(np.float32(v), np.float32(-np.inf)))
    rows = [[np.nan, 0, 0], [0, np.inf, 0], [0, 0, -np.inf], [2.5, 0, 0], [up(2.5), 0, 0],
            [0, 1.5, 0], [0, up(1.5), 0], [-2.5, -1.5, 0], [51.2, 0, 0], [below(51.2), 0, 0],
            [-51.2, 0, 0], [0, 0, 3.0], [0, 0, -5.0], [0.2, 0.2, 0.0], [0.4, 0.0, 0.0]]
    pts = np.zeros((len(rows), 5), np.float32)
    pts[:, :3] = rows
    pts[:, 3] = np.arange(len(rows)) / 16.0
    rois = [[0.0, 0.0, 2.0, 4.0, 0.0], [51.0, 0.0, 1.0, 1.0, 0.0], [-51.0, 0, 1, 1, 0]]
    w = _custom(pts, [0, len(rows)], [EYE], rois, margin=0.5)
    got, status, _ = run_gpu(mmbev_lib, w, cuda_dev)
    want = run_oracle(oracle_mod, w)
    assert status == 0
    assert_frames_equal(got, want, "boundaries")
    assert want[0][1].shape[0] >= 5


def test_duplicate_points_in_one_voxel(oracle_mod, mmbev_lib, cuda_dev):
    n = 5000
    pts = np.tile(np.array([[1.05, 2.05, 0.3, 0.5, 0.0]], np.float32), (n, 1))
    pts[:, 3] = (np.arange(n) % 32) / 32.0
    w = _custom(pts, [0, n], [EYE], FULL, K=10)
    got, status, _ = run_gpu(mmbev_lib, w, cuda_dev)
    assert status == 0
    assert got[0][2].tolist() == [10]
    assert_frames_equal(got, run_oracle(oracle_mod, w), "duplicates")


def test_tiny_grid_and_many_frames(oracle_mod, mmbev_lib, cuda_dev):
    # 4 x 3 x 2 = 24 cells (lins of five bits: one radix pass); 150 frames
    # of up to 60 points with 0..3 ROIs, so a compaction block's range holds
    # many frames (their counts and histograms go past the two it keeps in
    # shared memory), every frame is one sort tile, and max_voxels = 5 caps
    # most of them
    rng = np.random.default_rng(23)
    frames = []
    for f in range(150):
        n = int(rng.integers(0, 60))
        pts = np.zeros((n, 5), np.float32)
        pts[:, :3] = rng.uniform(-1, 1, (n, 3))
        pts[:, 3] = rng.uniform(0, 1, n)
        r = int(rng.integers(0, 4))
        rois = np.stack([rng.uniform(-1, 1, r), rng.uniform(-1, 1, r), rng.uniform(0.2, 1, r),
                         rng.uniform(0.2, 1, r), rng.uniform(0, 6, r)], 1) if r else np.zeros((0, 5))
        frames.append(_custom(pts, [0, n], [EYE], rois, margin=0.1, vs=(0.5, 2 / 3, 1.0),
                              rg=(-1, -1, -1, 1, 1, 1), K=2, maxv=5))
    b = synth.concat_frames(frames, "many")
    got, status, _ = run_gpu(mmbev_lib, b, cuda_dev)
    assert status == 0
    assert_frames_equal(got, run_oracle(oracle_mod, b), "many frames")


@pytest.mark.parametrize("K", [1, 64])
def test_grid_of_one_cell(oracle_mod, mmbev_lib, cuda_dev, K):
    # a 1 x 1 x 1 grid: every lin is 0, so no radix pass runs and the
    # compacted items, in input order, are already one run a frame; three
    # frames of 9,000 points span several sort and numbering tiles each
    rng = np.random.default_rng(25)
    frames = []
    for f in range(3):
        n = 9000
        pts = np.zeros((n, 5), np.float32)
        pts[:, :3] = rng.uniform(-0.99, 0.99, (n, 3))
        pts[:, 3] = rng.uniform(0, 1, n)
        pts[:, 4] = 0.05 * f
        frames.append(_custom(pts, [0, n], [EYE], FULL, vs=(2.0, 2.0, 2.0),
                              rg=(-1, -1, -1, 1, 1, 1), K=K))
    b = synth.concat_frames(frames, "one cell")
    got, status, _ = run_gpu(mmbev_lib, b, cuda_dev)
    assert status == 0
    want = run_oracle(oracle_mod, b)
    assert [w[2].tolist() for w in want] == [[K]] * 3
    assert assert_frames_equal(got, want, "one cell") == 1.0


def _max_frames_and_sweeps():
    # MMBEV_MAX_FRAMES frames of two sweeps each (MMBEV_MAX_SWEEPS sweeps),
    # the second sweep moved by a small turn and shift; up to 120 points a
    # sweep within 3 m, 0-4 rotated ROIs, K = 3 and max_voxels = 40
    rng = np.random.default_rng(26)
    frames = []
    for f in range(1024):
        n0, n1 = (int(x) for x in rng.integers(0, 121, 2))
        pts = np.zeros((n0 + n1, 5), np.float32)
        pts[:, :2] = rng.uniform(-3, 3, (n0 + n1, 2))
        pts[:, 2] = rng.uniform(-2, 2, n0 + n1)
        pts[:, 3] = rng.uniform(0, 1, n0 + n1)
        pts[n0:, 4] = 0.05
        a = rng.uniform(-0.05, 0.05)
        t1 = np.eye(4, dtype=np.float32)
        t1[:2, :2] = [[np.cos(a), -np.sin(a)], [np.sin(a), np.cos(a)]]
        t1[:2, 3] = rng.uniform(-0.5, 0.5, 2)
        r = int(rng.integers(0, 5))
        rois = np.stack([rng.uniform(-3, 3, r), rng.uniform(-3, 3, r), rng.uniform(0.5, 3, r),
                         rng.uniform(0.5, 3, r), rng.uniform(0, 6.3, r)], 1) if r else np.zeros((0, 5))
        frames.append(_custom(pts, [0, n0, n0 + n1], [EYE, t1.reshape(16)], rois, margin=0.2,
                              K=3, maxv=40))
    return synth.concat_frames(frames, "max frames")


def test_max_frames_and_sweeps(oracle_mod, mmbev_lib, cuda_dev):
    b = _max_frames_and_sweeps()
    assert b.num_frames == 1024 and len(b.sweep_offsets) == 2049
    got, status, _ = run_gpu(mmbev_lib, b, cuda_dev)
    assert status == 0
    assert assert_frames_equal(got, run_oracle(oracle_mod, b), "max frames") == 1.0


def test_max_rois_per_frame(oracle_mod, mmbev_lib, cuda_dev):
    # 1024 ROIs in a frame: 32 mask words per coarse cell
    rng = np.random.default_rng(24)
    r = 1024
    rois = np.stack([rng.uniform(-50, 50, r), rng.uniform(-50, 50, r), rng.uniform(0.5, 3, r),
                     rng.uniform(0.5, 6, r), rng.uniform(0, 6.3, r)], 1).astype(np.float32)
    w = synth.tiny(0).with_rois(rois)
    got, status, _ = run_gpu(mmbev_lib, w, cuda_dev)
    assert status == 0
    assert_frames_equal(got, run_oracle(oracle_mod, w), "1024 rois")
    assert got[0][1].shape[0] > 500


def test_single_frame_entry_equals_batched(oracle_mod, mmbev_lib, cuda_dev):
    w = synth.nuscenes_frame(5)
    pts, tf, rois = to_dev(w, cuda_dev)
    ws = mmbev_lib.new_workspace(w.num_points, w.rois.shape[0], w.max_voxels, 1, w.voxel_size,
                                 w.pc_range, cuda_dev)
    out = mmbev_lib.voxelize_roi(pts, w.sweep_offsets, tf, rois, w.roi_margin, w.voxel_size,
                                 w.pc_range, w.max_pts_per_voxel, w.max_voxels, workspace=ws)
    got = [out.frame(0, w.max_voxels)]
    assert mmbev_lib.get_status(ws) == 0
    assert_frames_equal(got, run_oracle(oracle_mod, w), "single-frame entry")


def test_repeat_calls_on_one_workspace_are_deterministic(mmbev_lib, cuda_dev):
    # the second call finds the first call's leftovers in the workspace
    w = synth.ouster_frame(2)
    a, s1, ws = run_gpu(mmbev_lib, w, cuda_dev)
    b, s2, _ = run_gpu(mmbev_lib, w, cuda_dev, workspace=ws)
    assert s1 == 0 and s2 == 0
    for (af, ac, an), (bf, bc, bn) in zip(a, b):
        assert np.array_equal(af.view(np.uint32), bf.view(np.uint32))
        assert np.array_equal(ac, bc) and np.array_equal(an, bn)


def test_non_default_stream(oracle_mod, mmbev_lib, cuda_dev):
    import torch
    w = synth.tiny(1)
    s = torch.cuda.Stream(cuda_dev)
    with torch.cuda.stream(s):
        got, status, _ = run_gpu(mmbev_lib, w, cuda_dev, stream=s)
    assert status == 0
    assert_frames_equal(got, run_oracle(oracle_mod, w), "stream")


def test_graph_capture_replays_the_call(oracle_mod, mmbev_lib, cuda_dev):
    import torch
    w = synth.nuscenes_frame(3)
    pts, tf, rois = to_dev(w, cuda_dev)
    ws = mmbev_lib.new_workspace(w.num_points, w.rois.shape[0], w.max_voxels, 1, w.voxel_size,
                                 w.pc_range, cuda_dev)
    out = mmbev_lib.Outputs.empty(1, w.max_voxels, cuda_dev)
    # one eager call first, as before any capture
    mmbev_lib.voxelize_roi_batched(pts, w.sweep_offsets, tf, rois, w.roi_margin, w.voxel_size,
                                   w.pc_range, w.max_pts_per_voxel, w.max_voxels,
                                   w.frame_sweep_offsets, w.frame_roi_offsets,
                                   workspace=ws, out=out)
    torch.cuda.synchronize()
    out.feats.zero_()
    out.coords.zero_()
    out.counts.zero_()
    out.nvox.zero_()
    torch.cuda.synchronize()
    g = torch.cuda.CUDAGraph()
    s = torch.cuda.Stream(cuda_dev)
    with torch.cuda.graph(g, stream=s):
        mmbev_lib.voxelize_roi_batched(pts, w.sweep_offsets, tf, rois, w.roi_margin, w.voxel_size,
                                       w.pc_range, w.max_pts_per_voxel, w.max_voxels,
                                       w.frame_sweep_offsets, w.frame_roi_offsets,
                                       workspace=ws, out=out)
    for _ in range(3):
        g.replay()
    torch.cuda.synchronize()
    assert mmbev_lib.get_status(ws) == 0
    assert_frames_equal([out.frame(0, w.max_voxels)], run_oracle(oracle_mod, w), "graph")


# ------------------------------------------------------------------ device-side failures

def test_reported_status_reaches_the_caller_and_clears(oracle_mod, mmbev_lib, cuda_dev):
    # A device-side failure is reported through the workspace's status word.
    # The test hook sets bits there as a failing kernel would (no kernel
    # fails): they reach mmbev_get_status, the call's results stay valid, and
    # the next call on the same workspace starts with a clear word.
    w = synth.nuscenes_frame(1)
    got, status, ws = run_gpu(mmbev_lib, w, cuda_dev,
                              inject_status=mmbev_lib.DEV_WAIT_TIMEOUT | mmbev_lib.DEV_BOUNDS)
    assert status == mmbev_lib.DEV_WAIT_TIMEOUT | mmbev_lib.DEV_BOUNDS
    assert_frames_equal(got, run_oracle(oracle_mod, w), "hooked call")
    _, status2, _ = run_gpu(mmbev_lib, synth.tiny(0), cuda_dev, workspace=ws)
    assert status2 == 0


def test_workspace_too_small_is_rejected(mmbev_lib, cuda_dev):
    import torch
    w = synth.tiny(0)
    pts, tf, rois = to_dev(w, cuda_dev)
    ws = torch.empty(4096, dtype=torch.uint8, device=cuda_dev)
    with pytest.raises(mmbev_lib.MMBEVError):
        mmbev_lib.voxelize_roi_batched(pts, w.sweep_offsets, tf, rois, 0.5, w.voxel_size,
                                       w.pc_range, 10, 16000, w.frame_sweep_offsets,
                                       w.frame_roi_offsets, workspace=ws)


# ------------------------------------------------------------------ rho_out (Alg. 1)

@pytest.mark.gpu
@pytest.mark.parametrize("rho", [0.1, 0.5, 1.0])
def test_rho_out_parity(oracle_mod, mmbev_lib, cuda_dev, rho):
    # points inside no ROI kept with probability rho (SplitMix64 draws), rank R_f
    w = synth.nuscenes_frame(1)
    got, status, _ = run_gpu(mmbev_lib, w, cuda_dev, rho_out=rho, seed=7)
    assert status == 0
    want = run_oracle(oracle_mod, w, rho_out=rho, seed=7)
    assert assert_frames_equal(got, want, f"rho={rho}") == 1.0


@pytest.mark.gpu
def test_rho_out_with_the_cap(oracle_mod, mmbev_lib, cuda_dev):
    # rho = 1 with a cap below the voxel count: background-only voxels (rank
    # R_f) go first, then the rank-tie split by lin
    w = synth.nuscenes_frame(1)
    for maxv in (9000, 30000):
        got, status, _ = run_gpu(mmbev_lib, w, cuda_dev, maxv=maxv, rho_out=1.0, seed=3)
        assert status == 0
        want = run_oracle(oracle_mod, w, maxv=maxv, rho_out=1.0, seed=3)
        assert len(want[0][1]) == maxv
        assert assert_frames_equal(got, want, f"rho cap {maxv}") == 1.0


@pytest.mark.gpu
def test_rho_out_batched_frames(oracle_mod, mmbev_lib, cuda_dev):
    # draws use frame-local indices: a batch equals its frames
    w = synth.concat_frames([synth.nuscenes_frame(s) for s in (1, 2, 3)], "three")
    got, status, _ = run_gpu(mmbev_lib, w, cuda_dev, rho_out=0.3, seed=12345)
    assert status == 0
    want = run_oracle(oracle_mod, w, rho_out=0.3, seed=12345)
    assert assert_frames_equal(got, want, "rho batch") == 1.0


@pytest.mark.gpu
def test_rho_out_seed_changes_the_draws(mmbev_lib, cuda_dev):
    w = synth.nuscenes_frame(1).with_rois(np.zeros((0, 5), np.float32))
    a, _, _ = run_gpu(mmbev_lib, w, cuda_dev, rho_out=0.5, seed=1)
    b, _, _ = run_gpu(mmbev_lib, w, cuda_dev, rho_out=0.5, seed=2)
    assert not np.array_equal(a[0][1], b[0][1])


# ------------------------------------------------------------------ ScatterToBEV (Alg. 1)

@pytest.mark.gpu
@pytest.mark.parametrize("name", ["tiny", "nuscenes_pillars"])
def test_scatter_bev_parity(oracle_mod, mmbev_lib, cuda_dev, name):
    import torch
    if name == "tiny":
        w = synth.tiny(0)
    else:  # the nuScenes frame on a pillar grid (0.075 x 0.075 x 8 m)
        base = synth.nuscenes_frame(1)
        w = synth.concat_frames([base, synth.nuscenes_frame(2)], "two")
        w.voxel_size = np.array([0.075, 0.075, 8.0], np.float32)
    got, status, _ = run_gpu(mmbev_lib, w, cuda_dev)
    assert status == 0
    want = run_oracle(oracle_mod, w)
    assert_frames_equal(got, want, name)
    dims = oracle_mod.grid_dims(w.voxel_size, w.pc_range)
    # the GPU scatter on the GPU voxelize outputs vs the oracle scatter of
    # the oracle's voxelize outputs
    pts, tf, rois = to_dev(w, cuda_dev)
    vx = mmbev_lib.Voxelizer(w.num_points, int(np.max(np.diff(w.frame_roi_offsets))), w.max_voxels,
                             w.num_frames, w.voxel_size, w.pc_range, w.max_pts_per_voxel,
                             w.roi_margin, device=cuda_dev)
    out = vx(pts, w.sweep_offsets, tf, rois, w.frame_sweep_offsets, w.frame_roi_offsets)
    canvas = mmbev_lib.scatter_bev(out, w.max_voxels, dims)
    torch.cuda.synchronize(cuda_dev)
    ref = oracle_mod.scatter_bev(want, dims)
    assert np.array_equal(canvas.cpu().numpy().view(np.uint32), ref.view(np.uint32))


@pytest.mark.gpu
def test_scatter_bev_refills_zeros_and_skips_bad_coords(oracle_mod, mmbev_lib, cuda_dev):
    import torch
    dims = (8, 4, 2)
    out = mmbev_lib.Outputs.empty(2, 3, device=cuda_dev)
    feats = torch.arange(30, dtype=torch.float32, device=cuda_dev).reshape(6, 5) + 1
    coords = torch.tensor([[0, 1, 2], [1, 3, 7], [0, 4, 0], [1, 0, 0], [5, 0, 0], [0, 0, 0]],
                          dtype=torch.int32, device=cuda_dev)   # row 2 and 4: outside dims
    out.feats.copy_(feats)
    out.coords.copy_(coords)
    out.nvox.copy_(torch.tensor([3, 2], dtype=torch.int32))
    canvas = torch.full((2, 10, 4, 8), 7.0, device=cuda_dev)    # stale contents get cleared
    mmbev_lib.scatter_bev(out, 3, dims, canvas=canvas)
    torch.cuda.synchronize(cuda_dev)
    f = feats.cpu().numpy()
    c = coords.cpu().numpy()
    frames = [(f[0:2], c[0:2], None), (f[3:4], c[3:4], None)]   # valid rows of each frame
    ref = oracle_mod.scatter_bev(frames, dims)
    assert np.array_equal(canvas.cpu().numpy(), ref)


# ------------------------------------------------------------------ temporal ROIs, criticality (Sec. IV-C)

CRIT = dict(v_ego=12.0, dt=0.1, a_brake=6.0, d_min=10.0, theta_max_deg=60.0, theta_min_deg=15.0,
            v_wide=5.0, v_narrow=30.0, tau_vru=1.5, tau_motor=2.5, r_coll=2.0)


def _random_objects(rng, n):
    o = np.zeros((n, 8), np.float32)
    o[:, 0] = rng.uniform(-40, 40, n)
    o[:, 1] = rng.uniform(-40, 40, n)
    o[:, 2] = rng.uniform(0.5, 3.0, n)
    o[:, 3] = rng.uniform(0.5, 6.0, n)
    o[:, 4] = rng.uniform(-np.pi, np.pi, n)
    o[:, 5] = rng.uniform(-15, 25, n)
    o[:, 6] = rng.uniform(-5, 5, n)
    o[:, 7] = rng.integers(0, 3, n)
    # a few exact ties in distance and TTC-free objects moving with the ego
    o[: n // 8, 5] = CRIT["v_ego"]
    o[: n // 8, 6] = 0.0
    if n > 4:
        o[1, :2] = o[0, :2]
    return o


@pytest.mark.gpu
def test_build_rois_parity(oracle_mod, mmbev_lib, cuda_dev):
    import torch
    rng = np.random.default_rng(21)
    counts = [0, 37, 512, 1, 200]
    objs = np.concatenate([_random_objects(rng, n) for n in counts]).astype(np.float32)
    off = np.concatenate([[0], np.cumsum(counts)]).astype(np.int32)
    for params in (CRIT, dict(CRIT, v_ego=0.0), dict(CRIT, v_ego=35.0, dt=0.0)):
        rois, flags, roff = mmbev_lib.build_rois(
            mmbev_lib.pack_objects(torch.from_numpy(objs).to(cuda_dev)), off, params)
        torch.cuda.synchronize(cuda_dev)
        rois, flags = rois.cpu().numpy(), flags.cpu().numpy()
        assert np.array_equal(roff, 2 * off)
        for f in range(len(counts)):
            want_r, want_f = oracle_mod.build_rois(objs[off[f]:off[f + 1]], params)
            assert np.array_equal(rois[2 * off[f]:2 * off[f + 1]].view(np.uint32), want_r.view(np.uint32))
            assert np.array_equal(flags[off[f]:off[f + 1]], want_f)


@pytest.mark.gpu
def test_built_rois_drive_the_voxelization(oracle_mod, mmbev_lib, cuda_dev):
    # the ROI table from the previous frame's detections feeds the call directly
    import torch
    frames = [synth.nuscenes_frame(s) for s in (1, 2)]
    rng = np.random.default_rng(5)
    objs = [_random_objects(rng, 40) for _ in frames]
    for o in objs:
        o[:, 0:2] = rng.uniform(-30, 30, (len(o), 2))
    allobj = np.concatenate(objs)
    off = np.array([0, 40, 80], np.int32)
    rois_d, _, roff = mmbev_lib.build_rois(
        mmbev_lib.pack_objects(torch.from_numpy(allobj).to(cuda_dev)), off, CRIT)
    w = synth.concat_frames([fw.with_rois(oracle_mod.build_rois(o, CRIT)[0])
                             for fw, o in zip(frames, objs)], "built")
    assert np.array_equal(w.frame_roi_offsets, roff)
    pts, tf, _ = to_dev(w, cuda_dev)
    vx = mmbev_lib.Voxelizer(w.num_points, 80, w.max_voxels, 2, w.voxel_size, w.pc_range,
                             w.max_pts_per_voxel, w.roi_margin, device=cuda_dev)
    out = vx(pts, w.sweep_offsets, tf, rois_d, w.frame_sweep_offsets, roff)
    torch.cuda.synchronize(cuda_dev)
    assert vx.status() == 0
    got = [out.frame(f, w.max_voxels) for f in range(2)]
    want = run_oracle(oracle_mod, w)
    assert assert_frames_equal(got, want, "built rois") == 1.0


# ------------------------------------------------------------------ voxel-grid components (proposer)

def _components_case(name):
    """(workload, per-frame voxel cap) of a components parity case."""
    if name == "tiny":
        return synth.tiny(0), None
    if name == "nuscenes":
        return synth.nuscenes_frame(1), None
    if name == "two_frames":
        return synth.concat_frames([synth.nuscenes_frame(s) for s in (1, 2)], "two"), None
    if name == "with_empty":   # a frame with no ROI (no kept voxel) between two
        return synth.concat_frames([synth.nuscenes_frame(1), synth.roi_coverage(0),
                                    synth.tiny(3)], "with_empty"), None
    if name == "multi_launch":   # a cap above 8 x 40,960 rows: the five-launch path
        return synth.concat_frames([synth.tiny(0), synth.tiny(5)], "two_tiny"), 400_000
    if name == "batch32":   # the full 32-frame batch, as the bench times it
        return synth.streaming_batch(32), None
    raise KeyError(name)


@pytest.mark.gpu
@pytest.mark.parametrize("name", ["tiny", "nuscenes", "two_frames", "with_empty", "multi_launch",
                                  "batch32"])
def test_voxel_components_parity(oracle_mod, mmbev_lib, cuda_dev, name):
    import torch
    w, maxv = _components_case(name)
    maxv = w.max_voxels if maxv is None else maxv
    pts, tf, rois = to_dev(w, cuda_dev)
    vx = mmbev_lib.Voxelizer(w.num_points, int(np.max(np.diff(w.frame_roi_offsets))), maxv,
                             w.num_frames, w.voxel_size, w.pc_range, w.max_pts_per_voxel,
                             w.roi_margin, device=cuda_dev)
    out = vx(pts, w.sweep_offsets, tf, rois, w.frame_sweep_offsets, w.frame_roi_offsets)
    dims = oracle_mod.grid_dims(w.voxel_size, w.pc_range)
    need = mmbev_lib.components_table_bytes(w.num_frames, maxv)
    table = torch.zeros(need, dtype=torch.uint8, device=cuda_dev) if need else None
    # twice on the same table: the first call must leave it all-zero
    for _ in range(2):
        labels, comp, ncomp, status = mmbev_lib.voxel_components(out, maxv, dims, table)
        torch.cuda.synchronize(cuda_dev)
        assert int(status.item()) == 0
        assert table is None or _table_is_clean(table)
    want = oracle_mod.voxel_components(run_oracle(oracle_mod, w, maxv=maxv), dims)
    labels, comp, ncomp = labels.cpu().numpy(), comp.cpu().numpy(), ncomp.cpu().numpy()
    nvox = out.nvox.cpu().numpy()
    for f, (wl, wc) in enumerate(want):
        r0 = f * maxv
        assert nvox[f] == len(wl)
        assert np.array_equal(labels[r0:r0 + nvox[f]], wl)
        assert np.all(labels[r0 + nvox[f]:r0 + maxv] == -1)
        assert ncomp[f] == len(wc)
        got = np.concatenate([wc[:, :1], comp[r0 + wc[:, 0]]], axis=1)
        assert np.array_equal(got, wc)


class _CoordsOut:
    """The two fields of a voxelize output that voxel_components reads."""
    def __init__(self, coords, nvox):
        self.coords, self.nvox = coords, nvox


@pytest.mark.gpu
def test_voxel_components_dense_blocks(oracle_mod, mmbev_lib, cuda_dev):
    """Solid blocks of voxels, rows in ascending index: every voxel has all 13
    earlier neighbours, and every CTA of the frame's cluster starts inside a
    block, so many pairs reach the previous CTA; plus isolated voxels and two
    blocks that touch only at a corner."""
    import torch
    dims = (1440, 1440, 40)   # (nx, ny, nz)
    cells = set()
    for z in range(2, 18):
        for y in range(100, 130):
            for x in range(200, 230):
                cells.add((z, y, x))
    for z in range(18, 22):   # a second block meeting the first at one corner
        for y in range(130, 140):
            for x in range(230, 240):
                cells.add((z, y, x))
    rng = np.random.default_rng(11)
    for _ in range(300):   # scattered voxels, mostly isolated
        cells.add((int(rng.integers(0, 40)), int(rng.integers(0, 1440)), int(rng.integers(0, 1440))))
    nx, ny, nz = dims
    coords = np.array(sorted(cells, key=lambda c: (c[0] * ny + c[1]) * nx + c[2]), np.int32)
    nv, maxv = len(coords), 20000
    assert nv <= maxv
    cbuf = np.zeros((maxv, 3), np.int32)
    cbuf[:nv] = coords
    out = _CoordsOut(torch.from_numpy(cbuf).to(cuda_dev),
                     torch.tensor([nv], dtype=torch.int32, device=cuda_dev))
    assert mmbev_lib.components_table_bytes(1, maxv) == 0   # the cluster path: no table
    labels, comp, ncomp, status = mmbev_lib.voxel_components(out, maxv, dims)
    torch.cuda.synchronize(cuda_dev)
    assert int(status.item()) == 0
    (wl, wc), = oracle_mod.voxel_components([(None, coords, None)], dims)
    labels = labels.cpu().numpy()
    assert np.array_equal(labels[:nv], wl)
    assert np.all(labels[nv:] == -1)
    assert int(ncomp.cpu()[0]) == len(wc)
    got = np.concatenate([wc[:, :1], comp.cpu().numpy()[wc[:, 0]]], axis=1)
    assert np.array_equal(got, wc)
    # the two blocks are one component (corner contact is 26-connected)
    row = {tuple(c): i for i, c in enumerate(coords.tolist())}
    assert labels[row[(2, 100, 200)]] == labels[row[(21, 139, 239)]]
    assert np.sum(labels[:nv] == labels[row[(2, 100, 200)]]) >= 30 * 30 * 16 + 4 * 10 * 10


@pytest.mark.gpu
def test_voxel_components_flags_unsorted_rows(mmbev_lib, cuda_dev):
    """Rows that do not ascend by linear index set MMBEV_DEV_UNSORTED."""
    import torch
    cbuf = np.array([[0, 0, 5], [0, 0, 2], [0, 0, 3], [0, 0, 0]], np.int32)
    out = _CoordsOut(torch.from_numpy(cbuf).to(cuda_dev),
                     torch.tensor([3], dtype=torch.int32, device=cuda_dev))
    _, _, _, status = mmbev_lib.voxel_components(out, 4, (8, 8, 1))
    torch.cuda.synchronize(cuda_dev)
    assert int(status.item()) & 0x8


@pytest.mark.gpu
@pytest.mark.parametrize("where", ["device", "pinned_host"])
def test_pack_voxels_gathers_every_frame(mmbev_lib, cuda_dev, where):
    """The packed buffer holds off[F+1] and every frame's kept rows in order,
    bit for bit, whether it lives on the device or in pinned host memory."""
    import torch
    w = synth.concat_frames([synth.nuscenes_frame(1), synth.roi_coverage(0), synth.tiny(3),
                             synth.nuscenes_frame(2)], "pack4")
    pts, tf, rois = to_dev(w, cuda_dev)
    vx = mmbev_lib.Voxelizer(w.num_points, int(np.max(np.diff(w.frame_roi_offsets))), w.max_voxels,
                             w.num_frames, w.voxel_size, w.pc_range, w.max_pts_per_voxel,
                             w.roi_margin, device=cuda_dev)
    out = vx(pts, w.sweep_offsets, tf, rois, w.frame_sweep_offsets, w.frame_roi_offsets)
    nbytes = mmbev_lib.pack_bytes(w.num_frames, w.max_voxels)
    if where == "device":
        dst = torch.full((nbytes,), 0xAB, dtype=torch.uint8, device=cuda_dev)
    else:
        dst = torch.full((nbytes,), 0xAB, dtype=torch.uint8).pin_memory()
    mmbev_lib.pack_voxels(out, w.max_voxels, dst)
    torch.cuda.synchronize(cuda_dev)
    off, feats, coords, counts = mmbev_lib.unpack(dst.cpu() if dst.is_cuda else dst, w.num_frames)
    off = off.numpy()
    nvox = out.nvox.cpu().numpy()
    assert off[0] == 0 and np.array_equal(np.diff(off), nvox)
    assert nvox[1] == 0   # the frame with no ROI
    for f in range(w.num_frames):
        ef, ec, en = out.frame(f, w.max_voxels)
        a, b = off[f], off[f + 1]
        assert np.array_equal(feats[a:b].numpy().view(np.uint32), ef.view(np.uint32))
        assert np.array_equal(coords[a:b].numpy(), ec)
        assert np.array_equal(counts[a:b].numpy(), en)
    # nothing written past the last record
    tail = (dst.cpu() if dst.is_cuda else dst)[4 * (w.num_frames + 1) + 36 * int(off[-1]):]
    assert bool((tail == 0xAB).all())


@pytest.mark.gpu
@pytest.mark.parametrize("chunk", [1, 3, 5, 8])
@pytest.mark.parametrize("rho", [0.0, 0.3])
def test_host_input_call_equals_device_input_call(mmbev_lib, cuda_dev, chunk, rho):
    """mmbev_voxelize_roi_batched_host (pinned host inputs, chunked copies on
    a side stream) gives exactly the outputs of the device-input call, for
    chunk sizes that do and do not divide the frame count."""
    import torch
    w = synth.concat_frames([synth.nuscenes_frame(s) for s in (1, 2, 3)] + [synth.roi_coverage(0)]
                            + [synth.tiny(s) for s in (4, 5)] + [synth.nuscenes_frame(6)],
                            "seven")
    pts, tf, rois = to_dev(w, cuda_dev)
    rmax = int(np.max(np.diff(w.frame_roi_offsets)))
    mk = lambda: mmbev_lib.Voxelizer(w.num_points, rmax, w.max_voxels, w.num_frames, w.voxel_size,
                                     w.pc_range, w.max_pts_per_voxel, w.roi_margin,
                                     device=cuda_dev, rho_out=rho, seed=9)
    ref = mk()
    want = ref(pts, w.sweep_offsets, tf, rois, w.frame_sweep_offsets, w.frame_roi_offsets)
    vx = mk()
    h_pts = torch.from_numpy(np.ascontiguousarray(w.points)).pin_memory()
    h_tf = torch.from_numpy(np.ascontiguousarray(w.sweep_tf)).pin_memory()
    h_rois = torch.from_numpy(np.ascontiguousarray(w.rois, np.float32).reshape(-1, 5)).pin_memory()
    nb = mmbev_lib.pack_bytes(w.num_frames, w.max_voxels)
    ref_pack = torch.zeros(nb, dtype=torch.uint8).pin_memory()
    mmbev_lib.pack_voxels(want, w.max_voxels, ref_pack)
    for it in range(2):   # twice: the staging is reused
        packed = torch.full((nb,), 0xCD, dtype=torch.uint8).pin_memory()
        got = vx.run_host(h_pts, w.sweep_offsets, h_tf, h_rois, w.frame_sweep_offsets,
                          w.frame_roi_offsets, chunk_frames=chunk,
                          pack_dst=packed if it == 1 else None)
        torch.cuda.synchronize(cuda_dev)
        assert vx.status() == 0
        assert torch.equal(got.nvox, want.nvox)
        if it == 1:   # packed chunk by chunk = packed in one go
            total = int(ref_pack[4 * w.num_frames:4 * w.num_frames + 4].view(torch.int32)[0])
            used = 4 * (w.num_frames + 1) + 36 * total
            assert torch.equal(packed[:used], ref_pack[:used])
            assert bool((packed[used:] == 0xCD).all())
        for f in range(w.num_frames):
            gf, gc, gn = got.frame(f, w.max_voxels)
            ef, ec, en = want.frame(f, w.max_voxels)
            assert np.array_equal(gf.view(np.uint32), ef.view(np.uint32))
            assert np.array_equal(gc, ec) and np.array_equal(gn, en)


@pytest.mark.gpu
def test_scatter_bev_update_equals_a_fresh_scatter(oracle_mod, mmbev_lib, cuda_dev):
    """A stream of frames through the update entry (previous cells cleared,
    new ones written) leaves, after every call, the canvas a fresh fill and
    scatter gives, bit for bit, and equal to the oracle's scatter."""
    import torch
    seqs = [[synth.nuscenes_frame(s) for s in (1, 2)], [synth.nuscenes_frame(s) for s in (3, 4)],
            [synth.roi_coverage(0), synth.nuscenes_frame(5)],
            [synth.nuscenes_frame(6), synth.nuscenes_frame(6)]]
    ws = [synth.concat_frames(fr, f"seq{i}") for i, fr in enumerate(seqs)]
    for w in ws:   # a pillar grid keeps the canvas small
        w.voxel_size = np.array([0.075, 0.075, 8.0], np.float32)
    w0 = ws[0]
    dims = oracle_mod.grid_dims(w0.voxel_size, w0.pc_range)
    rmax = max(int(np.max(np.diff(w.frame_roi_offsets))) for w in ws)
    npts = max(w.num_points for w in ws)
    vxs = [mmbev_lib.Voxelizer(npts, rmax, w0.max_voxels, 2, w0.voxel_size, w0.pc_range,
                               w0.max_pts_per_voxel, w0.roi_margin, device=cuda_dev)
           for _ in range(2)]                           # double-buffered outputs
    canvas = torch.zeros((2, dims[2] * 5, dims[1], dims[0]), device=cuda_dev)   # all-zero start
    prev = None
    for i, w in enumerate(ws):
        pts, tf, rois = to_dev(w, cuda_dev)
        out = vxs[i % 2](pts, w.sweep_offsets, tf, rois, w.frame_sweep_offsets,
                         w.frame_roi_offsets)
        mmbev_lib.scatter_bev_update(prev, out, w0.max_voxels, dims, canvas)
        fresh = mmbev_lib.scatter_bev(out, w0.max_voxels, dims)
        torch.cuda.synchronize(cuda_dev)
        assert torch.equal(canvas.view(torch.int32), fresh.view(torch.int32)), f"call {i}"
        ref = oracle_mod.scatter_bev(run_oracle(oracle_mod, w), dims)
        assert np.array_equal(canvas.cpu().numpy().view(np.uint32), ref.view(np.uint32))
        prev = out


@pytest.mark.gpu
def test_host_input_call_keeps_an_early_chunks_status(mmbev_lib, cuda_dev):
    """The workspace status accumulates over the chunks of a host-input call:
    a status bit set in the first chunk (the test hook, standing in for a
    device-side failure there) is still reported after the later chunks."""
    import torch
    w = synth.concat_frames([synth.nuscenes_frame(1), synth.tiny(2)], "big_then_small")
    rmax = int(np.max(np.diff(w.frame_roi_offsets)))
    vx = mmbev_lib.Voxelizer(w.num_points, rmax, w.max_voxels, w.num_frames, w.voxel_size,
                             w.pc_range, w.max_pts_per_voxel, w.roi_margin, device=cuda_dev)
    h_pts = torch.from_numpy(np.ascontiguousarray(w.points)).pin_memory()
    h_tf = torch.from_numpy(np.ascontiguousarray(w.sweep_tf)).pin_memory()
    h_rois = torch.from_numpy(np.ascontiguousarray(w.rois, np.float32).reshape(-1, 5)).pin_memory()
    vx.run_host(h_pts, w.sweep_offsets, h_tf, h_rois, w.frame_sweep_offsets, w.frame_roi_offsets,
                chunk_frames=1, inject_status=mmbev_lib.DEV_BOUNDS)
    torch.cuda.synchronize(cuda_dev)
    assert vx.status() == mmbev_lib.DEV_BOUNDS   # set in the first chunk only
    # the next call starts clean: the first chunk resets the status
    vx.run_host(h_pts, w.sweep_offsets, h_tf, h_rois, w.frame_sweep_offsets, w.frame_roi_offsets,
                chunk_frames=1)
    torch.cuda.synchronize(cuda_dev)
    assert vx.status() == 0


@pytest.mark.gpu
def test_back_to_back_host_calls_without_a_sync(mmbev_lib, cuda_dev):
    """Host-input calls issued back to back, with no synchronization between
    them: a call's uploads may overlap the previous call's work (the binding
    alternates two staging sets). Every call's packed rows equal those of the
    device-input call on the same inputs."""
    import torch
    ws = [synth.concat_frames([synth.nuscenes_frame(s), synth.nuscenes_frame(s + 1)], f"pair{s}")
          for s in (11, 21, 31)]
    w0 = ws[0]
    rmax = max(int(np.max(np.diff(w.frame_roi_offsets))) for w in ws)
    mk = lambda: mmbev_lib.Voxelizer(w0.num_points, rmax, w0.max_voxels, w0.num_frames,
                                     w0.voxel_size, w0.pc_range, w0.max_pts_per_voxel,
                                     w0.roi_margin, device=cuda_dev)
    nb = mmbev_lib.pack_bytes(w0.num_frames, w0.max_voxels)
    ref = mk()
    want = []
    for w in ws:
        pts, tf, rois = to_dev(w, cuda_dev)
        out = ref(pts, w.sweep_offsets, tf, rois, w.frame_sweep_offsets, w.frame_roi_offsets)
        buf = torch.zeros(nb, dtype=torch.uint8).pin_memory()
        mmbev_lib.pack_voxels(out, w0.max_voxels, buf)
        torch.cuda.synchronize(cuda_dev)
        want.append(buf)
    host = [tuple(torch.from_numpy(np.ascontiguousarray(a, np.float32).reshape(sh)).pin_memory()
                  for a, sh in ((w.points, (-1, 5)), (w.sweep_tf, (-1, 16)), (w.rois, (-1, 5))))
            for w in ws]
    vx = mk()
    got = [torch.full((nb,), 0xCD, dtype=torch.uint8).pin_memory() for _ in ws]
    for rnd in range(2):
        for w, (h_pts, h_tf, h_rois), dst in zip(ws, host, got):
            vx.run_host(h_pts, w.sweep_offsets, h_tf, h_rois, w.frame_sweep_offsets,
                        w.frame_roi_offsets, chunk_frames=1, pack_dst=dst)
        torch.cuda.synchronize(cuda_dev)
        assert vx.status() == 0
        for i, (g, e) in enumerate(zip(got, want)):
            total = int(e[4 * w0.num_frames:4 * w0.num_frames + 4].view(torch.int32)[0])
            used = 4 * (w0.num_frames + 1) + 36 * total
            assert torch.equal(g[:used], e[:used]), f"round {rnd}, call {i}"
