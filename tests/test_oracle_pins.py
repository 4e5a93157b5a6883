"""Pins of the oracle against facts that the paper and the mathematics fix.

Each group targets one step of the path and is built so that a plausible
slip in the oracle (a dropped term, a wrong sign, a transposed operand, a
swapped axis, the wrong half of an interval, the wrong K points) fails at
least one test. No expected value here comes from the code under test:
they follow from the construction of the inputs (voxel centres, exact
binary fractions, hand-placed ROIs), from an independent formulation
(double-precision polygon tests, a float64 matrix product) or from an
invariant of the definition.

Citations: Eq. 6-7 (motion compensation, Sec. IV-D), Eq. 1 (ROI boxes grown
by a margin, Sec. IV-C), Alg. 1 (inside-any-box keep, voxelize, voxel feature
encoder, Sec. IV-F), "hard voxelization" (per-voxel and per-frame caps,
Sec. IV-F), mandatory ROIs first (Sec. IV-C).
"""
import json
import os

import numpy as np
import pytest

import synth

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")

BIG_RANGE = np.array([-100.0, -100.0, -10.0, 100.0, 100.0, 10.0], np.float32)
ONE_VOXEL = np.array([200.0, 200.0, 20.0], np.float32)  # the whole range is one voxel


def eye_tf(n=1):
    return np.tile(np.eye(4, dtype=np.float32).reshape(1, 16), (n, 1))


def pts5(xyz, inten=None, dt=None):
    xyz = np.asarray(xyz, np.float32).reshape(-1, 3)
    p = np.zeros((xyz.shape[0], 5), np.float32)
    p[:, :3] = xyz
    if inten is not None:
        p[:, 3] = inten
    if dt is not None:
        p[:, 4] = dt
    return p


FULL_ROI = np.array([[0.0, 0.0, 1000.0, 1000.0, 0.0]], np.float32)


# ------------------------------------------------------------------ S1: Eq. 6-7

def test_identity_transform_is_exact(oracle_mod):
    rng = np.random.default_rng(1)
    p = pts5(rng.uniform(-60, 60, (500, 3)))
    xyz, _, _ = oracle_mod.classify(p, [0, 500], eye_tf(), FULL_ROI, 0.0, ONE_VOXEL, BIG_RANGE)
    assert np.array_equal(xyz, p[:, :3])


def test_translation_is_one_fp32_add(oracle_mod):
    rng = np.random.default_rng(2)
    p = pts5(rng.uniform(-60, 60, (500, 3)))
    tf = eye_tf()
    t = np.array([1.375, -20.3, 0.7], np.float32)
    tf[0, [3, 7, 11]] = t
    xyz, _, _ = oracle_mod.classify(p, [0, 500], tf, FULL_ROI, 0.0, ONE_VOXEL, BIG_RANGE)
    assert np.array_equal(xyz, p[:, :3] + t[None, :])


def test_quarter_turn_is_row_major_rotation(oracle_mod):
    # R = [[0,-1,0],[1,0,0],[0,0,1]] maps (x, y, z) to (-y, x, z); the
    # transposed reading would give (y, -x, z).
    rng = np.random.default_rng(3)
    p = pts5(rng.uniform(-60, 60, (300, 3)))
    tf = np.array([[0, -1, 0, 0, 1, 0, 0, 0, 0, 0, 1, 0, 0, 0, 0, 1]], np.float32)
    xyz, _, _ = oracle_mod.classify(p, [0, 300], tf, FULL_ROI, 0.0, ONE_VOXEL, BIG_RANGE)
    assert np.array_equal(xyz[:, 0], -p[:, 1])
    assert np.array_equal(xyz[:, 1], p[:, 0])
    assert np.array_equal(xyz[:, 2], p[:, 2])


def _rot(yaw, pitch, roll):
    cy, sy, cp, sp, cr, sr = (np.cos(yaw), np.sin(yaw), np.cos(pitch), np.sin(pitch),
                              np.cos(roll), np.sin(roll))
    rz = np.array([[cy, -sy, 0], [sy, cy, 0], [0, 0, 1]])
    ry = np.array([[cp, 0, sp], [0, 1, 0], [-sp, 0, cp]])
    rx = np.array([[1, 0, 0], [0, cr, -sr], [0, sr, cr]])
    return rz @ ry @ rx


def test_general_transform_within_fp32_rounding(oracle_mod):
    # Three rounded products and three rounded sums: the error is a few ulp of
    # the terms' magnitudes. Dropping any term or transposing R is off by far
    # more.
    rng = np.random.default_rng(4)
    n = 2000
    p = pts5(rng.uniform(-60, 60, (n, 3)))
    tfs, offs = [], [0]
    for s in range(4):
        m = np.eye(4)
        m[:3, :3] = _rot(*rng.uniform(-1.0, 1.0, 3))
        m[:3, 3] = rng.uniform(-20, 20, 3)
        tfs.append(m.astype(np.float32).reshape(16))
        offs.append(offs[-1] + n // 4)
    tf = np.stack(tfs)
    xyz, _, _ = oracle_mod.classify(p, offs, tf, FULL_ROI, 0.0, ONE_VOXEL, BIG_RANGE)
    for s in range(4):
        T = tf[s].astype(np.float64).reshape(4, 4)
        q = p[offs[s]:offs[s + 1], :3].astype(np.float64)
        exact = q @ T[:3, :3].T + T[:3, 3]
        mag = np.abs(q) @ np.abs(T[:3, :3]).T + np.abs(T[:3, 3])
        err = np.abs(xyz[offs[s]:offs[s + 1]] - exact)
        assert np.all(err <= 4 * np.finfo(np.float32).eps * mag + 1e-30)


def test_last_row_is_ignored(oracle_mod):
    rng = np.random.default_rng(5)
    p = pts5(rng.uniform(-60, 60, (200, 3)))
    tf = eye_tf()
    tf[0, [3, 7, 11]] = [1.0, 2.0, 3.0]
    tf2 = tf.copy()
    tf2[0, 12:16] = [7.0, -3.0, 0.5, 9.0]
    a, _, _ = oracle_mod.classify(p, [0, 200], tf, FULL_ROI, 0.0, ONE_VOXEL, BIG_RANGE)
    b, _, _ = oracle_mod.classify(p, [0, 200], tf2, FULL_ROI, 0.0, ONE_VOXEL, BIG_RANGE)
    assert np.array_equal(a, b)


def test_compensation_collapses_ghosts(oracle_mod):
    # Sec. IV-D: a static scene seen from several ego poses coincides after
    # compensation. Sensor-frame points are R_k^T (W - t_k); sweep_tf[k] is the
    # pose. The inverse convention would leave metre-scale ghosts.
    rng = np.random.default_rng(6)
    world = rng.uniform(-40, 40, (300, 3))
    pts, tfs, offs = [], [], [0]
    for k in range(10):
        px, py, yaw = -1.3 * k, 0.07 * k, 0.015 * k
        c, s = np.cos(yaw), np.sin(yaw)
        R = np.array([[c, -s, 0], [s, c, 0], [0, 0, 1]])
        local = (world - np.array([px, py, 0.0])) @ R  # R^T (W - t)
        pts.append(pts5(local))
        m = np.eye(4)
        m[:3, :3] = R
        m[:3, 3] = [px, py, 0.0]
        tfs.append(m.astype(np.float32).reshape(16))
        offs.append(offs[-1] + world.shape[0])
    p = np.concatenate(pts)
    xyz, _, _ = oracle_mod.classify(p, offs, np.stack(tfs), FULL_ROI, 0.0, ONE_VOXEL, BIG_RANGE)
    err = np.abs(xyz.reshape(10, -1, 3) - world[None]).max()
    assert err < 1e-4
    # and without compensation the copies are metres apart
    raw = p[:, :3].reshape(10, -1, 3)
    assert np.abs(raw[9] - world).max() > 1.0


# ------------------------------------------------------------------ S2: Alg. 1 / Eq. 1

def _corners(roi, margin):
    cx, cy, w, l, yaw = [float(v) for v in roi]
    hl, hw = 0.5 * l + margin, 0.5 * w + margin
    c, s = np.cos(yaw), np.sin(yaw)
    local = np.array([[hl, hw], [-hl, hw], [-hl, -hw], [hl, -hw]])  # counter-clockwise
    return np.stack([cx + c * local[:, 0] - s * local[:, 1],
                     cy + s * local[:, 0] + c * local[:, 1]], 1)


def _polygon_inside_and_edge_distance(px, py, corners):
    inside = np.ones(px.shape, bool)
    dmin = np.full(px.shape, np.inf)
    for k in range(4):
        a, b = corners[k], corners[(k + 1) % 4]
        ex, ey = b[0] - a[0], b[1] - a[1]
        cross = ex * (py - a[1]) - ey * (px - a[0])
        inside &= cross >= 0
        dmin = np.minimum(dmin, np.abs(cross) / np.hypot(ex, ey))
    return inside, dmin


def test_roi_membership_matches_polygon_bruteforce(oracle_mod):
    # Independent formulation: corners of the grown rectangle in double and a
    # point-in-convex-polygon test by cross products. Points within 1 mm of an
    # edge are left out (fp32 rounding decides those).
    rng = np.random.default_rng(7)
    n, r = 20000, 12
    p = pts5(np.stack([rng.uniform(-30, 30, n), rng.uniform(-30, 30, n),
                       rng.uniform(-1, 1, n)], 1))
    rois = np.stack([rng.uniform(-25, 25, r), rng.uniform(-25, 25, r), rng.uniform(0.5, 6, r),
                     rng.uniform(1, 12, r), rng.uniform(-np.pi, 2 * np.pi, r)], 1).astype(np.float32)
    margin = 0.75
    _, lin, rank = oracle_mod.classify(p, [0, n], eye_tf(), rois, margin, ONE_VOXEL, BIG_RANGE)
    px, py = p[:, 0].astype(np.float64), p[:, 1].astype(np.float64)
    expect = np.full(n, -1)
    near = np.zeros(n, bool)
    for k in range(r):
        ins, d = _polygon_inside_and_edge_distance(px, py, _corners(rois[k], margin))
        near |= d < 1e-3
        expect = np.where((expect < 0) & ins, k, expect)
    ok = ~near
    assert ok.sum() > 0.95 * n
    assert np.array_equal(rank[ok], expect[ok])
    assert np.array_equal(lin[ok] >= 0, expect[ok] >= 0)
    assert (expect >= 0).sum() > 500  # the test exercises hits, not only misses


def test_roi_boundary_is_inclusive_at_zero_yaw(oracle_mod):
    # Box at the origin, l = 4 along x, w = 2 along y, margin 0.5: the grown
    # half-extents are exactly 2.5 and 1.5.
    roi = np.array([[0.0, 0.0, 2.0, 4.0, 0.0]], np.float32)
    up = lambda v: np.nextafter(np.float32(v), np.float32(np.inf))
    xs = np.array([2.5, up(2.5), -2.5, -up(2.5), 0.0, 0.0, 0.0, 0.0, 2.5], np.float32)
    ys = np.array([0.0, 0.0, 0.0, 0.0, 1.5, up(1.5), -1.5, -up(1.5), 1.5], np.float32)
    want = np.array([0, -1, 0, -1, 0, -1, 0, -1, 0])
    p = pts5(np.stack([xs, ys, np.zeros_like(xs)], 1))
    _, _, rank = oracle_mod.classify(p, [0, len(xs)], eye_tf(), roi, 0.5, ONE_VOXEL, BIG_RANGE)
    assert np.array_equal(rank, want)


def test_length_runs_along_heading(oracle_mod):
    # yaw = pi/2: the 10 m length lies along +y, the 1 m width along x.
    roi = np.array([[0.0, 0.0, 1.0, 10.0, np.pi / 2]], np.float32)
    p = pts5([[0.0, 4.0, 0.0], [4.0, 0.0, 0.0], [0.0, -4.9, 0.0], [0.45, 0.0, 0.0]])
    _, _, rank = oracle_mod.classify(p, [0, 4], eye_tf(), roi, 0.0, ONE_VOXEL, BIG_RANGE)
    assert rank.tolist() == [0, -1, 0, 0]


def test_yaw_is_counter_clockwise(oracle_mod):
    # yaw = +30 deg: a point 4 m out along that heading is inside a 10 x 1 box,
    # the mirror point at -30 deg is not.
    a = np.deg2rad(30.0)
    roi = np.array([[0.0, 0.0, 1.0, 10.0, a]], np.float32)
    p = pts5([[4 * np.cos(a), 4 * np.sin(a), 0.0], [4 * np.cos(a), -4 * np.sin(a), 0.0]])
    _, _, rank = oracle_mod.classify(p, [0, 2], eye_tf(), roi, 0.0, ONE_VOXEL, BIG_RANGE)
    assert rank.tolist() == [0, -1]


def test_rank_is_first_containing_roi(oracle_mod):
    rois = np.array([[0.0, 0.0, 2.0, 2.0, 0.0],     # rank 0: |x|,|y| <= 1
                     [3.0, 0.0, 2.0, 8.0, 0.0],     # rank 1: -1 <= x <= 7
                     [0.0, 0.0, 20.0, 20.0, 0.0]],  # rank 2: everything near
                    np.float32)
    p = pts5([[0.5, 0.0, 0.0], [2.0, 0.0, 0.0], [9.0, 0.0, 0.0], [0.0, 9.5, 0.0],
              [30.0, 0.0, 0.0]])
    _, _, rank = oracle_mod.classify(p, [0, 5], eye_tf(), rois, 0.0, ONE_VOXEL, BIG_RANGE)
    assert rank.tolist() == [0, 1, 2, 2, -1]


def test_margin_grows_both_half_extents(oracle_mod):
    roi = np.array([[0.0, 0.0, 2.0, 4.0, 0.0]], np.float32)  # hl 2, hw 1 before the margin
    p = pts5([[2.9, 0.0, 0.0], [3.1, 0.0, 0.0], [0.0, 1.9, 0.0], [0.0, 2.1, 0.0]])
    _, _, rank = oracle_mod.classify(p, [0, 4], eye_tf(), roi, 1.0, ONE_VOXEL, BIG_RANGE)
    assert rank.tolist() == [0, -1, 0, -1]


def _trig_yaws(n_uniform, seed=7):
    """Yaws over several turns plus the multiples of pi/4 and their fp32
    neighbours (where cos and sin cross zero or meet each other)."""
    rng = np.random.default_rng(seed)
    u = rng.uniform(-8 * np.pi, 8 * np.pi, n_uniform).astype(np.float32)
    k = (np.arange(-32, 33) * (np.pi / 4)).astype(np.float32)
    near = [k]
    for steps in (1, 2, 3):
        near.append(np.nextafter(k, np.float32(np.inf)))
        near.append(np.nextafter(k, np.float32(-np.inf)))
        k = near[-2]
    return np.concatenate([u] + near).astype(np.float32)


def test_roi_box_trig_is_the_rounded_true_value(oracle_mod):
    # Eq. 1 box: the heading's cosine and sine, evaluated in double and
    # rounded to fp32. Checked against a 40-digit evaluation (mpmath): the
    # oracle's value must be the fp32 nearest to the true one, up to the
    # double-precision step before the rounding.
    mpmath = pytest.importorskip("mpmath")
    mpmath.mp.dps = 40
    yaws = _trig_yaws(20000)
    rois = np.zeros((yaws.size, 5), np.float32)
    rois[:, 2], rois[:, 3], rois[:, 4] = 2.0, 4.0, yaws
    box = oracle_mod.roi_boxes(rois, 0.5)
    for i, yaw in enumerate(yaws.tolist()):
        for col, fn in ((0, mpmath.cos), (1, mpmath.sin)):
            true = fn(mpmath.mpf(yaw))
            got = float(box[i, col])
            ulp = float(np.spacing(np.float32(abs(got)))) if got != 0.0 else 2.0 ** -149
            slack = 0.5 * ulp + 2.0 ** -52 * abs(float(true))
            assert abs(got - float(true)) <= slack, (yaw, col, got, float(true))
    assert np.all(box[:, 2] == 2.5) and np.all(box[:, 3] == 1.5)   # 0.5*4 + 0.5, 0.5*2 + 0.5


def test_no_rois_keeps_nothing(oracle_mod):
    w = synth.tiny(0)
    _, lin, _ = oracle_mod.classify(w.points, w.sweep_offsets, w.sweep_tf, w.rois[:0], 0.5,
                                    w.voxel_size, w.pc_range)
    assert (lin < 0).all()
    f, c, n = oracle_mod.voxelize_roi(w.points, w.sweep_offsets, w.sweep_tf, w.rois[:0], 0.5,
                                      w.voxel_size, w.pc_range, 10, 16000)
    assert len(n) == 0


def test_full_coverage_roi_keeps_every_in_range_point(oracle_mod):
    # Sec. IV-C fallback: with the ROI covering everything the path is plain
    # hard voxelization of the in-range points.
    w = synth.tiny(0)
    xyz, lin, rank = oracle_mod.classify(w.points, w.sweep_offsets, w.sweep_tf, FULL_ROI, 0.0,
                                         w.voxel_size, w.pc_range)
    rg = w.pc_range
    inr = np.ones(len(lin), bool)
    for a in range(3):
        inr &= (xyz[:, a] >= rg[a]) & (xyz[:, a] < rg[a + 3])
    assert np.array_equal(lin >= 0, inr)
    assert (rank[inr] == 0).all()


def test_range_is_half_open(oracle_mod):
    rg = np.array([-4.0, -4.0, -2.0, 4.0, 4.0, 2.0], np.float32)
    vs = np.array([1.0, 1.0, 1.0], np.float32)
    p = pts5([[-4.0, 0.0, 0.0], [4.0, 0.0, 0.0], [0.0, -4.0, 0.0], [0.0, 4.0, 0.0],
              [0.0, 0.0, -2.0], [0.0, 0.0, 2.0], [3.5, 3.5, 1.5]])
    _, lin, _ = oracle_mod.classify(p, [0, 7], eye_tf(), FULL_ROI, 0.0, vs, rg)
    assert (lin >= 0).tolist() == [True, False, True, False, True, False, True]


def test_index_rounding_onto_the_far_face_is_dropped(oracle_mod):
    # Just below xmax the point is in range, but (x - xmin) / size rounds up
    # to nx in fp32; such a point has no voxel and is dropped (c >= n rule).
    rg = np.array([-4.0, -4.0, -2.0, 4.0, 4.0, 2.0], np.float32)
    vs = np.array([1.0, 1.0, 1.0], np.float32)
    below = np.nextafter(np.float32(4.0), np.float32(0.0))
    assert np.float32(below - np.float32(-4.0)) / np.float32(1.0) == np.float32(8.0)
    p = pts5([[below, 0.0, 0.0], [0.0, below, 0.0], [3.75, 0.0, 0.0]])
    _, lin, _ = oracle_mod.classify(p, [0, 3], eye_tf(), FULL_ROI, 0.0, vs, rg)
    assert (lin >= 0).tolist() == [False, False, True]
    f, c, n = oracle_mod.voxelize_roi(p, [0, 3], eye_tf(), FULL_ROI, 0.0, vs, rg, 4, 10)
    assert c.tolist() == [[2, 4, 7]] and n.tolist() == [1]


def test_range_bound_inside_the_last_voxel(oracle_mod):
    # (max - min) / size = 16.5 rounds to 17 voxels, so the grid reaches 4.5
    # while the range stops at 4.25: points in [4.25, 4.5) have a voxel but are
    # out of range, and the range is half-open at 4.25.
    rg = np.array([-4.0, -4.0, -2.0, 4.25, 4.0, 2.0], np.float32)
    vs = np.array([0.5, 1.0, 1.0], np.float32)
    assert oracle_mod.grid_dims(vs, rg) == (17, 8, 4)
    p = pts5([[4.25, 0.0, 0.0], [4.3, 0.0, 0.0], [4.2, 0.0, 0.0]])
    _, lin, _ = oracle_mod.classify(p, [0, 3], eye_tf(), FULL_ROI, 0.0, vs, rg)
    assert (lin >= 0).tolist() == [False, False, True]
    f, c, n = oracle_mod.voxelize_roi(p, [0, 3], eye_tf(), FULL_ROI, 0.0, vs, rg, 4, 10)
    assert c.tolist() == [[2, 4, 16]]


def test_non_finite_points_are_dropped(oracle_mod):
    p = pts5([[np.nan, 0, 0], [0, np.inf, 0], [0, 0, -np.inf], [1.0, 1.0, 0.0]])
    _, lin, _ = oracle_mod.classify(p, [0, 4], eye_tf(), FULL_ROI, 0.0, ONE_VOXEL, BIG_RANGE)
    assert (lin >= 0).tolist() == [False, False, False, True]


def test_quarter_turn_invariance_of_membership(oracle_mod):
    rng = np.random.default_rng(8)
    n, r = 5000, 6
    xy = rng.uniform(-20, 20, (n, 2))
    p = pts5(np.stack([xy[:, 0], xy[:, 1], np.zeros(n)], 1))
    rois = np.stack([rng.uniform(-15, 15, r), rng.uniform(-15, 15, r), rng.uniform(1, 5, r),
                     rng.uniform(1, 8, r), rng.uniform(0, np.pi, r)], 1)
    q = pts5(np.stack([-xy[:, 1], xy[:, 0], np.zeros(n)], 1))
    rois_q = rois.copy()
    rois_q[:, 0], rois_q[:, 1], rois_q[:, 4] = -rois[:, 1], rois[:, 0], rois[:, 4] + np.pi / 2
    _, _, ra = oracle_mod.classify(p, [0, n], eye_tf(), rois.astype(np.float32), 0.3, ONE_VOXEL,
                                   BIG_RANGE)
    _, _, rb = oracle_mod.classify(q, [0, n], eye_tf(), rois_q.astype(np.float32), 0.3, ONE_VOXEL,
                                   BIG_RANGE)
    near = np.zeros(n, bool)
    for k in range(r):
        _, d = _polygon_inside_and_edge_distance(xy[:, 0], xy[:, 1], _corners(rois[k], 0.3))
        near |= d < 1e-3
    assert np.array_equal(ra[~near], rb[~near])
    assert (ra >= 0).sum() > 50


# ------------------------------------------------------------------ S3/S4: hard voxelization

GRID_RG = np.array([-8.0, -4.0, -2.0, 8.0, 4.0, 2.0], np.float32)
GRID_VS = np.array([0.25, 0.5, 1.0], np.float32)   # 64 x 16 x 4, all values binary fractions
NX, NY, NZ = 64, 16, 4


def _at(cx, cy, cz, fx=0.5, fy=0.5, fz=0.5):
    """Point at fraction (fx, fy, fz) inside voxel (cx, cy, cz)."""
    return [GRID_RG[0] + (cx + fx) * GRID_VS[0], GRID_RG[1] + (cy + fy) * GRID_VS[1],
            GRID_RG[2] + (cz + fz) * GRID_VS[2]]


def test_grid_dims(oracle_mod):
    assert oracle_mod.grid_dims(GRID_VS, GRID_RG) == (NX, NY, NZ)
    assert oracle_mod.grid_dims([0.075, 0.075, 0.2], [-54, -54, -5, 54, 54, 3]) == (1440, 1440, 40)


def test_voxel_index_by_construction(oracle_mod):
    rng = np.random.default_rng(9)
    c = np.stack([rng.integers(0, NX, 400), rng.integers(0, NY, 400), rng.integers(0, NZ, 400)], 1)
    centres = np.array([_at(*v) for v in c], np.float32)
    faces = np.array([_at(*v, 0.0, 0.0, 0.0) for v in c], np.float32)  # exact lower faces
    p = pts5(np.concatenate([centres, faces]))
    _, lin, _ = oracle_mod.classify(p, [0, len(p)], eye_tf(), FULL_ROI, 0.0, GRID_VS, GRID_RG)
    want = (c[:, 2] * NY + c[:, 1]) * NX + c[:, 0]   # z-major, then y, then x
    assert np.array_equal(lin, np.concatenate([want, want]))


def _dense_case(rng, n_vox, pts_per, K, maxv, rois=FULL_ROI, margin=0.0):
    """Random voxels, several points drawn strictly inside each, shuffled."""
    cells = rng.choice(NX * NY * NZ, n_vox, replace=False)
    cz, rem = np.divmod(cells, NX * NY)
    cy, cx = np.divmod(rem, NX)
    owner, xyz = [], []
    for v in range(n_vox):
        for _ in range(pts_per[v]):
            f = rng.uniform(0.05, 0.95, 3)
            xyz.append(_at(cx[v], cy[v], cz[v], *f))
            owner.append(v)
    owner = np.array(owner)
    perm = rng.permutation(len(owner))
    owner, xyz = owner[perm], np.array(xyz, np.float32)[perm]
    inten = rng.integers(0, 64, len(owner)) / 64.0
    dt = rng.integers(0, 8, len(owner)) * 0.125
    return pts5(xyz, inten, dt), owner, np.stack([cz, cy, cx], 1)


def test_dense_bucketing_first_k_and_order(oracle_mod):
    rng = np.random.default_rng(10)
    n_vox, K = 150, 3
    per = rng.integers(1, 7, n_vox)
    p, owner, zyx = _dense_case(rng, n_vox, per, K, 10**6)
    feats, coords, counts = oracle_mod.voxelize_roi(p, [0, len(p)], eye_tf(), FULL_ROI, 0.0,
                                                    GRID_VS, GRID_RG, K, 10**6)
    order = np.lexsort((zyx[:, 2], zyx[:, 1], zyx[:, 0]))   # by z, then y, then x
    assert np.array_equal(coords, zyx[order])
    for out_row, v in enumerate(order):
        idx = np.nonzero(owner == v)[0][:K]               # the K smallest input indices
        assert counts[out_row] == len(idx)
        want = p[idx].astype(np.float64).mean(0)
        np.testing.assert_allclose(feats[out_row], want, rtol=1e-6, atol=1e-6)


def test_sum_of_counts_invariant(oracle_mod):
    w = synth.nuscenes_frame(1)
    _, lin, _ = oracle_mod.classify(w.points, w.sweep_offsets, w.sweep_tf, w.rois, w.roi_margin,
                                    w.voxel_size, w.pc_range)
    n_v = np.unique(lin[lin >= 0], return_counts=True)[1]
    f, c, n = oracle_mod.voxelize_roi(w.points, w.sweep_offsets, w.sweep_tf, w.rois, w.roi_margin,
                                      w.voxel_size, w.pc_range, w.max_pts_per_voxel, w.max_voxels)
    assert len(n) == len(n_v)
    assert n.sum() == np.minimum(n_v, w.max_pts_per_voxel).sum()


def _cell_hits_roi(zyx, vs, rg, roi, margin):
    """Separating-axis test, in double, of a voxel's BEV cell against a grown ROI."""
    x0 = rg[0] + zyx[2] * vs[0]
    y0 = rg[1] + zyx[1] * vs[1]
    cell = np.array([[x0, y0], [x0 + vs[0], y0], [x0 + vs[0], y0 + vs[1]], [x0, y0 + vs[1]]])
    rect = _corners(roi, margin)
    for poly in (cell, rect):
        for k in range(4):
            e = poly[(k + 1) % 4] - poly[k]
            ax = np.array([-e[1], e[0]])
            a, b = cell @ ax, rect @ ax
            if a.max() < b.min() - 1e-6 or b.max() < a.min() - 1e-6:
                return False
    return True


def test_every_voxel_touches_an_roi(oracle_mod):
    w = synth.nuscenes_frame(1)
    f, c, n = oracle_mod.voxelize_roi(w.points, w.sweep_offsets, w.sweep_tf, w.rois, w.roi_margin,
                                      w.voxel_size, w.pc_range, w.max_pts_per_voxel, w.max_voxels)
    vs, rg = w.voxel_size.astype(np.float64), w.pc_range.astype(np.float64)
    rng = np.random.default_rng(11)
    for row in rng.choice(len(c), 400, replace=False):
        assert any(_cell_hits_roi(c[row], vs, rg, roi, w.roi_margin) for roi in w.rois)


def test_adding_rois_never_removes_voxels(oracle_mod):
    w = synth.roi_coverage(32)
    kw = dict(voxel_size=w.voxel_size, pc_range=w.pc_range, max_pts_per_voxel=10,
              max_voxels=10**6)
    a = oracle_mod.voxelize_roi(w.points, w.sweep_offsets, w.sweep_tf, w.rois[:10], w.roi_margin, **kw)
    b = oracle_mod.voxelize_roi(w.points, w.sweep_offsets, w.sweep_tf, w.rois, w.roi_margin, **kw)
    sa = {tuple(r) for r in a[1]}
    sb = {tuple(r) for r in b[1]}
    assert sa and sa <= sb and len(sb) > len(sa)


def test_cap_keeps_smallest_rank_then_smallest_lin(oracle_mod):
    # Eight voxels, U = max_voxels + 3. Row (cz=1, cy=3) holds cx 10, 11, 40,
    # 41, 50, 60; row (cz=1, cy=9) holds cx 20, 30. ROI 0 covers cx 38..62 of
    # row 3 (four voxels), ROI 1 covers cx 5..15 of row 3 (two voxels), ROI 2
    # covers row 9. With max_voxels = 5 all four rank-0 voxels stay and, of the
    # two rank-1 voxels, only the one with the smaller lin (cx 10). Voxel 11's
    # point comes first in the input, so a first-seen rule would keep it.
    def box(cx0, cx1, cy):
        x0 = GRID_RG[0] + cx0 * GRID_VS[0]
        x1 = GRID_RG[0] + (cx1 + 1) * GRID_VS[0]
        y = GRID_RG[1] + (cy + 0.5) * GRID_VS[1]
        return [0.5 * (x0 + x1), y, 0.2, x1 - x0 - 0.1, 0.0]
    rois = np.array([box(38, 62, 3), box(5, 15, 3), box(0, 63, 9)], np.float32)
    order = [(11, 3), (10, 3), (40, 3), (41, 3), (50, 3), (60, 3), (20, 9), (30, 9)]
    p = pts5([_at(cx, cy, 1) for cx, cy in order])
    _, _, rank = oracle_mod.classify(p, [0, len(p)], eye_tf(), rois, 0.0, GRID_VS, GRID_RG)
    assert rank.tolist() == [1, 1, 0, 0, 0, 0, 2, 2]
    f, coords, counts = oracle_mod.voxelize_roi(p, [0, len(p)], eye_tf(), rois, 0.0, GRID_VS,
                                                GRID_RG, 4, 5)
    assert coords.tolist() == [[1, 3, 10], [1, 3, 40], [1, 3, 41], [1, 3, 50], [1, 3, 60]]
    # room for seven: both rank-1 voxels, one of the rank-2 ones (smaller lin)
    f, coords, counts = oracle_mod.voxelize_roi(p, [0, len(p)], eye_tf(), rois, 0.0, GRID_VS,
                                                GRID_RG, 4, 7)
    assert coords[:, 2].tolist() == [10, 11, 40, 41, 50, 60, 20]


def test_cap_uses_minimum_rank_of_the_voxels_points(oracle_mod):
    # Voxel A holds a rank-2 point and a rank-0 point (minimum 0); voxel B only
    # rank-1 points. With room for one voxel, A is kept although its first
    # point has the worse rank.
    a0 = _at(5, 5, 1, 0.2, 0.5, 0.5)
    a1 = _at(5, 5, 1, 0.8, 0.5, 0.5)
    b0 = _at(2, 5, 1)
    rois = np.array([[a1[0], a1[1], 0.05, 0.05, 0.0],   # rank 0: only a1
                     [b0[0], b0[1], 0.2, 0.2, 0.0],     # rank 1: b0
                     [a0[0], a0[1], 0.05, 0.05, 0.0]],  # rank 2: only a0
                    np.float32)
    p = pts5([a0, b0, a1])
    f, coords, counts = oracle_mod.voxelize_roi(p, [0, 3], eye_tf(), rois, 0.0, GRID_VS, GRID_RG,
                                                4, 1)
    assert coords.tolist() == [[1, 5, 5]]
    assert counts.tolist() == [2]


def test_max_voxels_zero_gives_nothing(oracle_mod):
    w = synth.tiny(0)
    f, c, n = oracle_mod.voxelize_roi(w.points, w.sweep_offsets, w.sweep_tf, w.rois, w.roi_margin,
                                      w.voxel_size, w.pc_range, 10, 0)
    assert len(n) == 0


# ------------------------------------------------------------------ S5: voxel feature encoder

def test_single_point_voxel_mean_is_the_point(oracle_mod):
    tf = eye_tf()
    tf[0, [3, 7, 11]] = [0.5, -0.25, 0.125]
    p = pts5([_at(10, 2, 1)], [0.375], [0.25])
    p[:, :3] -= np.array([0.5, -0.25, 0.125], np.float32)
    f, c, n = oracle_mod.voxelize_roi(p, [0, 1], tf, FULL_ROI, 0.0, GRID_VS, GRID_RG, 10, 100)
    assert c.tolist() == [[1, 2, 10]] and n.tolist() == [1]
    assert np.array_equal(f[0], np.array(_at(10, 2, 1) + [0.375, 0.25], np.float32))


def test_k1_keeps_the_lowest_index(oracle_mod):
    rng = np.random.default_rng(12)
    xyz = [_at(7, 7, 2, *rng.uniform(0.1, 0.9, 3)) for _ in range(6)]
    p = pts5(xyz, np.arange(6) / 8.0, 0.0)
    f, c, n = oracle_mod.voxelize_roi(p, [0, 6], eye_tf(), FULL_ROI, 0.0, GRID_VS, GRID_RG, 1, 10)
    assert n.tolist() == [1]
    assert np.array_equal(f[0], p[0])


def test_first_ten_of_twelve_by_index_across_sweeps(oracle_mod):
    # 12 points of one voxel spread over two sweeps, interleaved with points
    # of other voxels; intensities are binary fractions so every sum is exact.
    rng = np.random.default_rng(13)
    target = []
    rows = []
    for i in range(40):
        if i % 3 == 0 and len(target) < 12:
            rows.append(_at(30, 8, 2, *rng.uniform(0.1, 0.9, 3)))
            target.append(i)
        else:
            rows.append(_at(int(rng.integers(0, 20)), 1, 0, *rng.uniform(0.1, 0.9, 3)))
    inten = (np.arange(40) % 16) / 16.0
    p = pts5(rows, inten, np.where(np.arange(40) < 20, 0.0, 0.5))
    tf = eye_tf(2)
    f, c, n = oracle_mod.voxelize_roi(p, [0, 20, 40], tf, FULL_ROI, 0.0, GRID_VS, GRID_RG, 10, 100)
    row = [k for k, v in enumerate(c.tolist()) if v == [2, 8, 30]][0]
    first10 = target[:10]
    assert n[row] == 10
    assert f[row, 3] == np.float32(inten[first10].sum()) / np.float32(10)
    assert f[row, 4] == np.float32(np.where(np.array(first10) < 20, 0.0, 0.5).sum()) / np.float32(10)
    np.testing.assert_allclose(f[row, :3], p[first10, :3].astype(np.float64).mean(0), rtol=1e-6)


# ------------------------------------------------------------------ batched form

def test_batched_equals_independent_frames(oracle_mod):
    frames = [synth.tiny(s) for s in range(3)]
    b = synth.concat_frames(frames, "tiny3")
    outs = oracle_mod.voxelize_roi_batched(b.points, b.sweep_offsets, b.sweep_tf, b.rois,
                                           b.roi_margin, b.voxel_size, b.pc_range,
                                           b.max_pts_per_voxel, b.max_voxels,
                                           b.frame_sweep_offsets, b.frame_roi_offsets)
    for w, (f, c, n) in zip(frames, outs):
        ef, ec, en = oracle_mod.voxelize_roi(w.points, w.sweep_offsets, w.sweep_tf, w.rois,
                                             w.roi_margin, w.voxel_size, w.pc_range,
                                             w.max_pts_per_voxel, w.max_voxels)
        assert np.array_equal(c, ec) and np.array_equal(n, en) and np.array_equal(f, ef)
    assert sum(len(o[2]) for o in outs) > 0


# ------------------------------------------------------------------ stored regression value

def test_tiny_matches_stored_oracle_output(oracle_mod):
    """tests/golden/tiny_seed0.json was written by tests/golden/make_golden.py,
    which calls only the oracle; it guards the oracle against silent drift."""
    with open(os.path.join(GOLDEN, "tiny_seed0.json")) as fh:
        g = json.load(fh)
    w = synth.tiny(0)
    f, c, n = oracle_mod.voxelize_roi(w.points, w.sweep_offsets, w.sweep_tf, w.rois, w.roi_margin,
                                      w.voxel_size, w.pc_range, w.max_pts_per_voxel, w.max_voxels)
    assert c.tolist() == g["coords"]
    assert n.tolist() == g["counts"]
    assert [[float.hex(float(v)) for v in row] for row in f] == g["feats_hex"]


# ------------------------------------------------------------------ rho_out (Alg. 1)

def _vox(oracle_mod, w, rho_out=0.0, seed=0, max_pts_per_voxel=None, max_voxels=None):
    return oracle_mod.voxelize_roi(
        w.points, w.sweep_offsets, w.sweep_tf, w.rois, w.roi_margin, w.voxel_size, w.pc_range,
        w.max_pts_per_voxel if max_pts_per_voxel is None else max_pts_per_voxel,
        w.max_voxels if max_voxels is None else max_voxels, rho_out=rho_out, seed=seed)


def test_splitmix64_matches_the_published_stream(oracle_mod):
    # pins the counter-based generator that decides out-of-ROI keeps
    ref = json.load(open(os.path.join(GOLDEN, "splitmix64_seed0.json")))
    got = [oracle_mod.splitmix64(ref["seed"], n + 1) for n in range(len(ref["outputs"]))]
    assert got == [int(h, 16) for h in ref["outputs"]]


def _frame_without_rois():
    w = synth.nuscenes_frame(1)
    return w.with_rois(np.zeros((0, 5), np.float32))


def test_rho_zero_keeps_only_roi_points(oracle_mod):
    w = synth.nuscenes_frame(1)
    a = _vox(oracle_mod, w)
    b = _vox(oracle_mod, w, rho_out=0.0, seed=99)
    for x, y in zip(a, b):
        assert np.array_equal(x.view(np.uint32), y.view(np.uint32))


def test_rho_one_is_dense_voxelization(oracle_mod):
    # every in-range point kept: the same output as one box covering the range
    w = _frame_without_rois()
    dense = synth.roi_coverage("full")
    got = _vox(oracle_mod, w, rho_out=1.0, seed=5)
    want = _vox(oracle_mod, dense)
    for x, y in zip(got, want):
        assert np.array_equal(x.view(np.uint32), y.view(np.uint32))


def test_rho_below_one_draw_keeps_nothing(oracle_mod):
    # floor(rho * 2^24) = 0: no draw can pass
    w = _frame_without_rois()
    f, c, n = _vox(oracle_mod, w, rho_out=1e-9, seed=5)
    assert len(c) == 0


def test_background_keep_fraction_follows_rho(oracle_mod):
    w = _frame_without_rois()
    dense = synth.roi_coverage("full")
    big = dict(max_pts_per_voxel=1 << 20, max_voxels=1 << 20)
    in_range = int(_vox(oracle_mod, dense, **big)[2].sum())
    for rho in (0.1, 0.5):
        kept = int(_vox(oracle_mod, w, rho_out=rho, seed=11, **big)[2].sum())
        sd = np.sqrt(in_range * rho * (1 - rho))
        assert abs(kept - rho * in_range) < 5 * sd, (rho, kept, in_range)


def test_background_voxels_rank_below_every_roi(oracle_mod):
    # capped to the voxels that hold an ROI point, rho = 1 keeps exactly them
    w = synth.nuscenes_frame(1)
    roi_only = _vox(oracle_mod, w)
    u = len(roi_only[1])
    got = _vox(oracle_mod, w, rho_out=1.0, seed=3, max_voxels=u)
    assert np.array_equal(got[1], roi_only[1])
    full = _vox(oracle_mod, w, rho_out=1.0, seed=3)
    assert len(full[1]) > u


def test_draws_use_frame_local_indices(oracle_mod):
    frames = [synth.nuscenes_frame(s) for s in (1, 2)]
    b = synth.concat_frames(frames, "two")
    out = oracle_mod.voxelize_roi_batched(
        b.points, b.sweep_offsets, b.sweep_tf, b.rois, b.roi_margin, b.voxel_size, b.pc_range,
        b.max_pts_per_voxel, b.max_voxels, b.frame_sweep_offsets, b.frame_roi_offsets,
        rho_out=0.25, seed=17)
    for fw, got in zip(frames, out):
        want = _vox(oracle_mod, fw, rho_out=0.25, seed=17)
        for x, y in zip(got, want):
            assert np.array_equal(x.view(np.uint32), y.view(np.uint32))


# ------------------------------------------------------------------ ScatterToBEV (Alg. 1)

def test_scatter_bev_places_features_by_coordinate(oracle_mod):
    feats = np.array([[1, 2, 3, 4, 5], [6, 7, 8, 9, 10]], np.float32)
    coords = np.array([[0, 2, 3], [1, 0, 1]], np.int32)   # (z, y, x)
    canvas = oracle_mod.scatter_bev([(feats, coords, np.array([1, 1], np.int32))], (4, 3, 2))
    assert canvas.shape == (1, 10, 3, 4)
    assert list(canvas[0, 0:5, 2, 3]) == [1, 2, 3, 4, 5]
    assert list(canvas[0, 5:10, 0, 1]) == [6, 7, 8, 9, 10]
    assert np.count_nonzero(canvas) == 10


def test_scatter_bev_pillars_is_the_bev_map(oracle_mod):
    # nz = 1: channel c of cell (cy, cx) is feature c; the canvas sums to the features
    w = synth.tiny(0)
    out = oracle_mod.voxelize_roi(w.points, w.sweep_offsets, w.sweep_tf, w.rois, w.roi_margin,
                                  w.voxel_size, w.pc_range, w.max_pts_per_voxel, w.max_voxels)
    dims = oracle_mod.grid_dims(w.voxel_size, w.pc_range)
    canvas = oracle_mod.scatter_bev([out], dims)
    feats, coords, _ = out
    assert canvas.shape == (1, 5, dims[1], dims[0])
    assert np.allclose(canvas.sum(axis=(0, 2, 3), dtype=np.float64), feats.sum(0, dtype=np.float64))
    occupied = np.count_nonzero(np.any(canvas[0] != 0, axis=0))
    assert occupied <= len(coords)
    for v in (0, len(coords) // 2, len(coords) - 1):
        assert np.array_equal(canvas[0, :, coords[v, 1], coords[v, 2]], feats[v])


# ------------------------------------------------------------------ temporal ROIs, criticality (Sec. IV-C)

CRIT = dict(v_ego=10.0, dt=0.1, a_brake=6.0, d_min=10.0, theta_max_deg=60.0, theta_min_deg=15.0,
            v_wide=5.0, v_narrow=30.0, tau_vru=1.5, tau_motor=2.5, r_coll=2.0)


def _obj(cx, cy, vx=0.0, vy=0.0, cls=0, w=2.0, l=4.5, yaw=0.0):
    return [cx, cy, w, l, yaw, vx, vy, cls]


def test_braking_distance_and_cone(oracle_mod):
    # Eq. 4: dmax = max(d_min, v^2 / (2 a)); the cone half-angle spans 60 .. 15 deg
    d, t = oracle_mod.crit_thresholds(dict(CRIT, v_ego=10.0))
    assert d == pytest.approx(10.0) and t == pytest.approx(np.tan(np.radians(51.0)), rel=1e-6)
    d, t = oracle_mod.crit_thresholds(dict(CRIT, v_ego=20.0))
    assert d == pytest.approx(400.0 / 12.0, rel=1e-6)
    assert oracle_mod.crit_thresholds(dict(CRIT, v_ego=0.0))[1] == pytest.approx(np.sqrt(3), rel=1e-6)
    assert oracle_mod.crit_thresholds(dict(CRIT, v_ego=40.0))[1] == pytest.approx(
        np.tan(np.radians(15.0)), rel=1e-6)


def test_time_to_collision_closed_forms(oracle_mod):
    # ego at 10 m/s: a parked car 20 m ahead closes at 10 m/s, t* = 2 s
    objs = np.array([_obj(20, 0, cls=0), _obj(20, 0, cls=1), _obj(20, 5, cls=0),
                     _obj(20, 0, vx=15.0, cls=0), _obj(20, 0, cls=2)], np.float32)
    _, flags = oracle_mod.build_rois(objs, CRIT)
    assert flags[0] == 2          # Safety: TTC 2 <= 2.5 (motorized)
    assert flags[1] == 0          # VRU threshold 1.5 < 2
    assert flags[2] == 0          # passes 5 m to the side: beyond r_coll
    assert flags[3] == 0          # pulling away: t* < 0
    assert flags[4] == 0          # static: geometry only, and it is out of the cone range


def test_geometry_cone_is_inclusive_and_forward(oracle_mod):
    d, t = oracle_mod.crit_thresholds(CRIT)
    x = np.float32(5.0)
    y_edge = np.float32(x * np.float32(t))
    objs = np.array([_obj(x, y_edge, vx=10.0), _obj(x, np.nextafter(y_edge, np.float32(1e9)), vx=10.0),
                     _obj(-1.0, 0.0, vx=10.0), _obj(9.9, 0.0, vx=10.0), _obj(10.1, 0.0, vx=10.0)],
                    np.float32)   # vx = v_ego: no relative motion, no TTC
    _, flags = oracle_mod.build_rois(objs, CRIT)
    assert list(flags) == [1, 0, 0, 1, 0]


def test_ranking_mandatory_then_ttc_then_distance(oracle_mod):
    objs = np.array([_obj(30, 20, vx=10.0),            # optional, far
                     _obj(3, 1, vx=10.0),              # optional? in the cone and near: Geom
                     _obj(20, 0, cls=0),               # Safety, TTC 2.0
                     _obj(15, 0, cls=0),               # Safety, TTC 1.5
                     _obj(8, 25, vx=10.0)], np.float32)   # optional, nearer than the first
    rois, flags = oracle_mod.build_rois(objs, CRIT)
    order = [int(np.argmin(np.abs(objs[:, 0] - r[0]) + np.abs(objs[:, 1] - r[1]))) for r in rois[::2]]
    # mandatory (TTC 1.5, TTC 2.0, then the Geom-only one with TTC inf), then optional by distance
    assert order == [3, 2, 1, 4, 0]
    assert list(flags) == [0, 1, 2, 2, 0]


def test_each_object_gives_its_box_and_the_extrapolated_box(oracle_mod):
    objs = np.array([_obj(12.0, -3.0, vx=4.0, vy=1.5, cls=1, w=0.8, l=0.9, yaw=0.3)], np.float32)
    rois, _ = oracle_mod.build_rois(objs, CRIT)
    assert rois.shape == (2, 5)
    assert list(rois[0]) == [12.0, -3.0, 0.8, 0.9, np.float32(0.3)]
    rvx, rvy = np.float32(4.0 - 10.0), np.float32(1.5)
    assert rois[1][0] == np.float32(12.0) + rvx * np.float32(0.1)
    assert rois[1][1] == np.float32(-3.0) + rvy * np.float32(0.1)
    assert list(rois[1][2:]) == list(rois[0][2:])


# ------------------------------------------------------------------ voxel-grid components (proposer)

def _cc(oracle_mod, coords, dims=(16, 16, 4)):
    coords = np.asarray(coords, np.int32).reshape(-1, 3)
    feats = np.zeros((len(coords), 5), np.float32)
    return oracle_mod.voxel_components([(feats, coords, None)], dims)[0]


def test_components_use_26_connectivity(oracle_mod):
    # face, edge and corner neighbours join; a gap of one cell separates
    labels, comp = _cc(oracle_mod, [[0, 0, 0], [0, 0, 1], [0, 1, 2], [1, 2, 3], [1, 2, 5]])
    assert list(labels) == [0, 0, 0, 0, 4]
    assert comp.tolist() == [[0, 4, 0, 0, 0, 1, 2, 3], [4, 1, 1, 2, 5, 1, 2, 5]]


def test_component_label_is_the_smallest_row(oracle_mod):
    # rows listed out of spatial order: the label is the smallest row index
    labels, comp = _cc(oracle_mod, [[0, 5, 5], [0, 9, 9], [0, 5, 6], [0, 9, 8], [0, 5, 7]])
    assert list(labels) == [0, 1, 0, 1, 0]
    assert comp[:, 0].tolist() == [0, 1] and comp[:, 1].tolist() == [3, 2]


def test_component_sizes_sum_to_the_voxels(oracle_mod):
    w = synth.nuscenes_frame(1)
    out = _vox(oracle_mod, w)
    dims = oracle_mod.grid_dims(w.voxel_size, w.pc_range)
    labels, comp = oracle_mod.voxel_components([out], dims)[0]
    assert comp[:, 1].sum() == len(out[1])
    assert np.all(labels[comp[:, 0]] == comp[:, 0])   # roots label themselves
    assert np.all(labels <= np.arange(len(labels)))


@pytest.mark.parametrize("density", [0.05, 0.2, 0.45])
def test_components_match_textbook_26_connected_labelling(oracle_mod, density):
    """The partition, sizes and boxes equal scipy.ndimage.label with a full
    3x3x3 structuring element (26-connectivity) on a small dense grid."""
    ndimage = pytest.importorskip("scipy.ndimage")
    rng = np.random.default_rng(int(density * 100))
    nz, ny, nx = 6, 14, 17
    occ = rng.random((nz, ny, nx)) < density
    zs, ys, xs = np.nonzero(occ)                       # ascending linear index
    coords = np.stack([zs, ys, xs], 1).astype(np.int32)
    perm = rng.permutation(len(coords))                # rows in any order
    coords = coords[perm]
    labels, comp = _cc(oracle_mod, coords, dims=(nx, ny, nz))
    ref, nref = ndimage.label(occ, structure=np.ones((3, 3, 3), bool))
    ref_of_row = ref[coords[:, 0], coords[:, 1], coords[:, 2]]
    assert len(comp) == nref
    # same partition: the map oracle label -> scipy label is a bijection
    pairs = set(zip(labels.tolist(), ref_of_row.tolist()))
    assert len(pairs) == nref
    assert len({p[0] for p in pairs}) == nref and len({p[1] for p in pairs}) == nref
    # each label is the smallest row of its component
    for lab in np.unique(labels):
        assert lab == np.min(np.nonzero(labels == lab)[0])
    # sizes and bounding boxes
    for row in comp:
        lab, size = int(row[0]), int(row[1])
        r = ref_of_row[lab]
        cz, cy, cx = np.nonzero(ref == r)
        assert size == len(cz)
        assert row[2:].tolist() == [cz.min(), cy.min(), cx.min(), cz.max(), cy.max(), cx.max()]
