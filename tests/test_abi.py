"""The C-ABI library builds for sm_103a, loads without a GPU, exports every
entry point include/mmbev.h declares, and rejects bad host arguments before
touching the device."""
import ctypes
import os
import re

import numpy as np
import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "mmbev.h")

TINY_VS = np.array([0.2, 0.2, 8.0], np.float32)
TINY_RG = np.array([-51.2, -51.2, -5.0, 51.2, 51.2, 3.0], np.float32)


def declared_functions():
    text = open(HEADER).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(mmbev_[a-z_]+)\s*\(", text)))


def test_header_declares_the_boundary():
    names = declared_functions()
    for required in ("mmbev_voxelize_roi", "mmbev_voxelize_roi_batched", "mmbev_workspace_size",
                     "mmbev_classify_points", "mmbev_get_status", "mmbev_prep_rois"):
        assert required in names


def test_library_exports_every_declared_symbol(mmbev_lib):
    lib = mmbev_lib.load()
    missing = [n for n in declared_functions() if not hasattr(lib, n)]
    assert not missing, missing


def test_sizes_are_host_only(mmbev_lib):
    a = mmbev_lib.workspace_size(20000, 4, 16000, 1, TINY_VS, TINY_RG)
    b = mmbev_lib.workspace_size(40000, 4, 16000, 1, TINY_VS, TINY_RG)
    c = mmbev_lib.workspace_size(20000, 4, 16000, 2, TINY_VS, TINY_RG)
    assert 0 < a < b and a < c
    with pytest.raises(ValueError):
        mmbev_lib.workspace_size(20000, 4, 16000, 1, TINY_VS, [0, 0, 0, -1, 1, 1])



def test_workspace_size_follows_the_documented_rule(mmbev_lib):
    # about 66 bytes a point plus about 34 KB a frame; max_voxels does not
    # enter; the no-alloc array then holds about 1.5 M points of one frame
    vs = np.array([0.075, 0.075, 0.2], np.float32)
    rg = np.array([-54, -54, -5, 54, 54, 3], np.float32)
    ws = lambda n, mv=120000, F=1: mmbev_lib.workspace_size(n, 30, mv, F, vs, rg)
    per_point = (ws(2_000_000) - ws(1_000_000)) / 1_000_000
    assert 65.5 <= per_point <= 66.5
    assert 32_000 <= ws(1000, F=2) - ws(1000) <= 35_000
    assert ws(1_000_000, 1) == ws(1_000_000, 200_000)
    m = re.search(r"#define MMBEV_NOALLOC_SCRATCH_BYTES \((\d+)u << (\d+)\)", open(HEADER).read())
    cap = int(m.group(1)) << int(m.group(2))
    assert ws(1_450_000) <= cap < ws(1_600_000)

def _call(lib, *, so=(0, 100), fso=None, fro=None, nr=1, K=10, maxv=100, vs=TINY_VS, rg=TINY_RG,
          margin=0.5, ws_bytes=1 << 30, ws=0x7f0000000000):
    so = np.asarray(so, np.int64)
    ns = len(so) - 1
    fso = np.asarray([0, ns] if fso is None else fso, np.int32)
    fro = np.asarray([0, nr] if fro is None else fro, np.int32)
    vs = np.asarray(vs, np.float32)
    rg = np.asarray(rg, np.float32)
    P = ctypes.c_void_p
    fake = P(0x7e0000000000)  # never dereferenced: validation fails first
    return lib.mmbev_voxelize_roi_batched(
        fake, so.ctypes.data_as(P), ns, fake, fake, nr, margin, vs.ctypes.data_as(P),
        rg.ctypes.data_as(P), K, maxv, len(fso) - 1, fso.ctypes.data_as(P), fro.ctypes.data_as(P),
        fake, fake, fake, fake, P(ws), ws_bytes, None)


@pytest.mark.parametrize("kw", [
    dict(K=0), dict(K=65), dict(maxv=-1), dict(so=(1, 100)), dict(so=(0, 50, 40)),
    dict(fso=(0, 2)), dict(fro=(0, 2)), dict(margin=-0.1), dict(margin=float("nan")),
    dict(vs=(0.2, 0.0, 8.0)), dict(rg=(0, 0, 0, 0, 1, 1)), dict(rg=(0, 0, 0, float("inf"), 1, 1)),
    dict(ws=0x7f0000000010), dict(nr=2000, fro=(0, 2000)),
    dict(vs=(1e-4, 1e-4, 1e-4)),   # more than 2^32 cells
    dict(so=[0] * 2050),            # too many sweeps
])
def test_invalid_arguments_are_rejected_before_launch(mmbev_lib, kw):
    assert _call(mmbev_lib.load(), **kw) == -1


def test_small_buffers_are_rejected_before_launch(mmbev_lib):
    lib = mmbev_lib.load()
    assert _call(lib, ws_bytes=1024) == -3


def _max_points():
    m = re.search(r"#define MMBEV_MAX_POINTS\s+(\d+)LL", open(HEADER).read())
    return int(m.group(1))


def test_point_limit_keeps_record_slots_below_2_32(mmbev_lib):
    # whole 2,048-point tiles of record slots below 2^32: the largest call
    # passes validation (and needs far more than the 1 GB workspace given);
    # one point more is invalid, and so is its workspace size
    lim = _max_points()
    assert lim % 2048 == 0 and lim + 2048 == 1 << 32
    lib = mmbev_lib.load()
    assert _call(lib, so=(0, lim)) == -3
    assert _call(lib, so=(0, lim + 1)) == -1
    assert mmbev_lib.workspace_size(lim, 4, 16000, 1, TINY_VS, TINY_RG) > 66 * lim
    with pytest.raises(ValueError):
        mmbev_lib.workspace_size(lim + 1, 4, 16000, 1, TINY_VS, TINY_RG)


@pytest.mark.parametrize("rho", [-0.1, 1.5, float("nan")])
def test_rho_out_outside_unit_interval_is_rejected(mmbev_lib, rho):
    lib = mmbev_lib.load()
    so = np.asarray((0, 100), np.int64)
    fso = np.asarray([0, 1], np.int32)
    fro = np.asarray([0, 1], np.int32)
    P = ctypes.c_void_p
    fake = P(0x7e0000000000)
    opts = mmbev_lib._ExecOpts(None, 0, rho, 1)
    rc = lib.mmbev_voxelize_roi_batched_ex(
        fake, so.ctypes.data_as(P), 1, fake, fake, 1, 0.5, TINY_VS.ctypes.data_as(P),
        TINY_RG.ctypes.data_as(P), 10, 100, 1, fso.ctypes.data_as(P), fro.ctypes.data_as(P),
        fake, fake, fake, fake, P(0x7f0000000000), 1 << 30, None, ctypes.byref(opts))
    assert rc == -1


def test_scatter_bev_checks_the_canvas(mmbev_lib):
    lib = mmbev_lib.load()
    P = ctypes.c_void_p
    fake = P(0x7e0000000000)
    dims = np.asarray([512, 512, 1], np.int32)
    need = 2 * 512 * 512 * 5 * 4
    args = (fake, fake, fake, 2, 100, dims.ctypes.data_as(P))
    assert lib.mmbev_scatter_bev(*args, P(0x7f0000000000), need - 16, None) == -3
    assert lib.mmbev_scatter_bev(*args, P(0x7f0000000004), need, None) == -1
    bad = np.asarray([512, 0, 1], np.int32)
    assert lib.mmbev_scatter_bev(fake, fake, fake, 2, 100, bad.ctypes.data_as(P),
                                 P(0x7f0000000000), need, None) == -1


def test_build_rois_validates_on_the_host(mmbev_lib):
    lib = mmbev_lib.load()
    P = ctypes.c_void_p
    fake = P(0x7e0000000000)
    good = dict(v_ego=10.0, dt=0.1, a_brake=6.0, d_min=10.0, theta_max_deg=60.0,
                theta_min_deg=15.0, v_wide=5.0, v_narrow=30.0, tau_vru=1.5, tau_motor=2.5,
                r_coll=2.0)

    def call(off, **kw):
        q = np.asarray([float(dict(good, **kw)[k]) for k in mmbev_lib.CRIT_FIELDS], np.float32)
        off = np.asarray(off, np.int32)
        return lib.mmbev_build_rois(fake, off.ctypes.data_as(P), len(off) - 1,
                                    q.ctypes.data_as(P), fake, fake, None)
    assert call([0, 513]) == -1                 # more objects than half the ROI limit
    assert call([0, 5, 3]) == -1                # offsets decrease
    assert call([1, 5]) == -1                   # must start at 0
    assert call([0, 5], a_brake=0.0) == -1
    assert call([0, 5], v_narrow=4.0) == -1
    assert call([0, 5], dt=float("nan")) == -1
    assert call([0, 0]) == 0                    # nothing to do: no launch


def test_workspace_size_is_monotone_in_the_roi_count(mmbev_lib):
    # a workspace sized for up to R ROIs per frame serves every call with fewer
    sizes = [mmbev_lib.workspace_size(20000, r, 16000, 4, TINY_VS, TINY_RG)
             for r in (1, 32, 33, 64, 128, 129, 512, 1024)]
    assert sizes == sorted(sizes)


def test_voxel_components_checks_the_table(mmbev_lib):
    lib = mmbev_lib.load()
    P = ctypes.c_void_p
    fake = P(0x7e0000000000)
    dims = np.asarray([512, 512, 1], np.int32)
    # caps up to 8 x 32,768 rows take the cluster path: no table
    assert lib.mmbev_components_table_size(2, 16000) == 0
    assert lib.mmbev_components_table_size(1, 262144) == 0
    # larger caps: per frame 2^k >= 4 * cap slots of 8 bytes, then the scratch
    maxv = 300000
    H = 1 << 21
    need = 2 * H * 8 + 4 * 2 * maxv
    assert lib.mmbev_components_table_size(2, maxv) == need
    assert lib.mmbev_components_table_size(-1, 10) == 0
    assert lib.mmbev_components_table_size(1, (1 << 28) + 1) == 0
    args = (fake, fake, 2, maxv, dims.ctypes.data_as(P))
    tail = (fake, fake, fake, None, None)
    assert lib.mmbev_voxel_components(*args, P(0x7f1000000000), need - 4, *tail) == -3
    assert lib.mmbev_voxel_components(*args, P(0x7f1000000008), need, *tail) == -1
    assert lib.mmbev_voxel_components(*args, None, need, *tail) == -1
    bad = np.asarray([512, 512, 0], np.int32)
    assert lib.mmbev_voxel_components(fake, fake, 2, 16000, bad.ctypes.data_as(P),
                                      None, 0, *tail) == -1
    assert lib.mmbev_voxel_components(fake, fake, 2, (1 << 28) + 1, dims.ctypes.data_as(P),
                                      None, 0, *tail) == -1



def test_pack_voxels_checks_its_arguments(mmbev_lib):
    lib = mmbev_lib.load()
    P = ctypes.c_void_p
    fake = P(0x7e0000000000)
    # off[F+1] then 36 bytes a row of the cap
    assert lib.mmbev_pack_size(2, 1000) == 4 * 3 + 36 * 2 * 1000
    assert lib.mmbev_pack_size(0, 1000) == 4
    assert lib.mmbev_pack_size(-1, 10) == 0
    need = lib.mmbev_pack_size(2, 1000)
    args = (fake, fake, fake, fake, 2, 1000)
    assert lib.mmbev_pack_voxels(*args, P(0x7f2000000000), need - 4, None) == -3
    assert lib.mmbev_pack_voxels(*args, P(0x7f2000000002), need, None) == -1   # not 4-byte aligned
    assert lib.mmbev_pack_voxels(*args, None, need, None) == -1
    assert lib.mmbev_pack_voxels(fake, fake, fake, fake, -1, 1000, P(0x7f2000000000), need,
                                 None) == -1


def test_host_input_call_checks_offsets_before_copying(mmbev_lib):
    lib = mmbev_lib.load()
    P = ctypes.c_void_p
    fake = P(0x7e0000000000)
    vs = np.asarray([0.2, 0.2, 8.0], np.float32)
    rg = np.asarray([-51.2, -51.2, -5.0, 51.2, 51.2, 3.0], np.float32)
    so = np.asarray([0, 100, 250], np.int64)

    def call(fso, fro, chunk=1, nsw=2, nroi=3, so=so):
        fso = np.asarray(fso, np.int32)
        fro = np.asarray(fro, np.int32)
        return lib.mmbev_voxelize_roi_batched_host(
            fake, so.ctypes.data_as(P), nsw, fake, fake, nroi, 0.5, vs.ctypes.data_as(P),
            rg.ctypes.data_as(P), 10, 1000, len(fso) - 1, fso.ctypes.data_as(P),
            fro.ctypes.data_as(P), fake, fake, fake, fake, fake, fake, fake, fake, 1 << 20,
            None, 0, chunk, None, None, None)

    assert call([0, 1, 2], [0, 1, 3], chunk=0) == -1           # chunk_frames < 1
    assert call([1, 1, 2], [0, 1, 3]) == -1                     # frames must start at sweep 0
    assert call([0, 1, 3], [0, 1, 3]) == -1                     # last frame past the sweeps
    assert call([0, 2, 1], [0, 1, 3], nsw=1) == -1              # decreasing
    assert call([0, 1, 2], [0, 2, 1], nroi=1) == -1             # decreasing ROI offsets
    assert call([0, 1, 2], [0, 1, 3], so=np.asarray([0, 100, 50], np.int64)) == -1


def test_scatter_bev_update_checks_its_arguments(mmbev_lib):
    lib = mmbev_lib.load()
    P = ctypes.c_void_p
    fake = P(0x7e0000000000)
    dims = np.asarray([100, 50, 2], np.int32)
    need = 2 * 100 * 50 * 2 * 5 * 4
    args = (fake, fake, fake, 2, 10, dims.ctypes.data_as(P))
    assert lib.mmbev_scatter_bev_update(fake, fake, *args, P(0x7f3000000000), need - 4, None) == -3
    assert lib.mmbev_scatter_bev_update(fake, fake, *args, P(0x7f3000000004), need, None) == -1
    assert lib.mmbev_scatter_bev_update(fake, None, *args, P(0x7f3000000000), need, None) == -1
    bad = np.asarray([100, 0, 2], np.int32)
    assert lib.mmbev_scatter_bev_update(None, None, fake, fake, fake, 2, 10, bad.ctypes.data_as(P),
                                        P(0x7f3000000000), need, None) == -1


def test_stage_names_follow_the_launch_order(mmbev_lib):
    # one name per kernel of a call, in launch order; out of range: empty
    names = mmbev_lib.stage_names()
    assert names == ["prep", "classify", "compact", "sort", "runs", "emit"]
    lib = mmbev_lib.load()
    assert lib.mmbev_stage_name(mmbev_lib.NUM_STAGES) == b""
    assert lib.mmbev_stage_name(-1) == b""
    text = open(HEADER).read()
    assert re.search(r"#define MMBEV_NUM_STAGES\s+%d\b" % mmbev_lib.NUM_STAGES, text)
