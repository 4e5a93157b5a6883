/*
 * mmbev.h -- C ABI of the GB300 (sm_103a) ROI-aware multi-sweep LiDAR
 * voxelization library (MM-BEV, arXiv 2608.15437).
 *
 * The library computes, for one or many independent frames, the LiDAR hot
 * path of the paper's sparse ROI-aware feature extraction:
 *
 *   S1  per-sweep ego-motion compensation, p' = R p + T          (Sec. IV-D, Eq. 6-7)
 *   S2  range crop and inside-any-ROI test against criticality-ranked,
 *       margin-grown rotated BEV boxes, then the voxel index        (Alg. 1; Eq. 1)
 *   S3  voxel dedup                                                 (Alg. 1, "Voxelize")
 *   S4  voxel cap and canonical (ascending linear index) order      (Sec. IV-F "hard
 *                                                                    voxelization"; Sec. IV-C)
 *   S5  mean features over the first K points of each voxel         (Alg. 1, "VoxelFeatureEncoder")
 *
 * Exact semantics (every GPU result equals this, bit for bit for integers
 * and, by construction, for the fp32 features too):
 *   - Point i of sweep s (sweep_offsets[s] <= i < sweep_offsets[s+1]) with
 *     T = sweep_tf[s] (row-major 4x4, last row ignored, sweep frame -> current
 *     frame): x' = ((T0*x + T1*y) + T2*z) + T3, likewise y' (T4..T7) and
 *     z' (T8..T11); every fp32 product and sum rounded on its own (no FMA).
 *   - Range: xmin <= x' < xmax, same for y and z (NaN and Inf fail).
 *   - ROI r (cx, cy, w, l, yaw): c = (float)cos((double)yaw),
 *     s = (float)sin((double)yaw), hl = 0.5f*l + margin, hw = 0.5f*w + margin,
 *     dx = x'-cx, dy = y'-cy, u = dx*c + dy*s, v = dy*c - dx*s; inside iff
 *     |u| <= hl and |v| <= hw. l runs along the heading, w across it, yaw is
 *     counter-clockwise from +x. The point's rank is the first ROI (in array
 *     order = criticality order) that contains it; a point in no ROI is
 *     dropped, except that mmbev_voxelize_roi_batched_ex can keep such points
 *     at the rate rho_out of Alg. 1 (see mmbev_exec_opts_t).
 *   - Voxel: c_a = (int)floorf((p'_a - min_a) / size_a), dropped if
 *     c_a >= n_a, with n_a = (int)llround(((double)max_a - min_a) / size_a);
 *     lin = (cz*ny + cy)*nx + cx.
 *   - Each voxel keeps its K = max_pts_per_voxel points with the smallest
 *     input index. If a frame has more than max_voxels voxels, the
 *     max_voxels smallest by (minimum rank of the voxel's points, lin) are
 *     kept. Kept voxels are written in ascending lin.
 *   - feats = (x', y', z', intensity, dt) summed in fp32 over the kept points
 *     in index order, divided once by (float)count.
 *
 * Execution model. Every call is asynchronous on `stream`: it validates its
 * host arguments, enqueues a fixed sequence of kernels and returns. It never
 * synchronizes, never allocates and reads its host arrays only during the
 * call, so it can be captured in a CUDA graph. The caller owns every buffer.
 *
 * One caller-owned device buffer, the `workspace` (size from
 * mmbev_workspace_size), is the library's scratch. It carries no state from
 * one call to the next, except the device status word that
 * mmbev_get_status reads; any contents are fine on entry. Calls that share
 * a workspace must not overlap on the GPU.
 *
 * Errors. A status below zero is returned before any launch when a host
 * argument is invalid (MMBEV_EINVAL) or a buffer is too small
 * (MMBEV_EWORKSPACE), and after a failed launch (MMBEV_ECUDA). Conditions
 * only the device can see (an internal wait that timed out, an internal
 * index out of its bounds) set bits in a device status word instead; no
 * kernel traps or spins without bound. mmbev_get_status reads it. After a
 * non-zero device status the outputs are invalid; the next call starts
 * afresh.
 */
#ifndef MMBEV_H_
#define MMBEV_H_

#include <stddef.h>
#include <stdint.h>
#include <cuda_runtime_api.h>

#ifdef __cplusplus
extern "C" {
#endif

/* One BEV region of interest in the current ego frame: centre (cx, cy) in
 * metres, width w (lateral) and length l (along the heading) in metres,
 * heading yaw in radians, counter-clockwise from +x. This is the box of
 * Eq. 1; the margin r of Eq. 1 is passed separately (roi_margin) and grows
 * both half-extents. */
typedef struct mmbev_roi {
    float cx, cy, w, l, yaw;
} mmbev_roi_t;

typedef enum mmbev_status {
    MMBEV_OK = 0,
    MMBEV_EINVAL = -1,      /* invalid host argument; nothing launched */
    MMBEV_ECUDA = -2,       /* a CUDA runtime call or launch failed */
    MMBEV_EWORKSPACE = -3   /* workspace or another buffer smaller than required */
} mmbev_status_t;

/* Device status bits (mmbev_get_status). */
#define MMBEV_DEV_TABLE_FULL   0x1u  /* components: a voxel key found no free slot */
#define MMBEV_DEV_WAIT_TIMEOUT 0x2u  /* an internal inter-block wait gave up */
#define MMBEV_DEV_BOUNDS       0x4u  /* an internal index failed its bounds check */
#define MMBEV_DEV_UNSORTED     0x8u  /* components: a frame's rows do not ascend by linear index */

/* Limits of one call. */
#define MMBEV_MAX_SWEEPS          2048
#define MMBEV_MAX_FRAMES          1024
#define MMBEV_MAX_ROIS_PER_FRAME  1024
#define MMBEV_MAX_PTS_PER_VOXEL   64
/* 2^32 - 2,048 points: the record slots, a whole number of 2,048-point
 * tiles, keep 32-bit positions. */
#define MMBEV_MAX_POINTS          4294965248LL

/*
 * Bytes of scratch workspace for a call with up to max_points points,
 * max_rois_per_frame ROIs in any frame, max_voxels kept voxels per frame and
 * num_frames frames on the grid given by voxel_size[3] and range[6] (host
 * arrays). About 66 bytes per point (records, sort keys and positions and
 * per-voxel results, all sized for every point kept) plus about 34 KB per
 * frame. Returns 0 for invalid arguments (max_points above MMBEV_MAX_POINTS
 * among them).
 */
size_t mmbev_workspace_size(int64_t max_points, int32_t max_rois_per_frame,
                            int32_t max_voxels, int32_t num_frames,
                            const float voxel_size[3], const float range[6]);

/*
 * One frame (Alg. 1 on the union of n sweeps, Eq. 7).
 *   points         device, float32 [N][5] (x, y, z, intensity, dt), 16-byte
 *                  aligned; N = sweep_offsets[num_sweeps] <= MMBEV_MAX_POINTS.
 *   sweep_offsets  host, int64 [num_sweeps+1], sweep_offsets[0] = 0,
 *                  nondecreasing; sweep s owns points [off[s], off[s+1]).
 *   num_sweeps     0 <= num_sweeps <= MMBEV_MAX_SWEEPS.
 *   sweep_tf       device, float32 [num_sweeps][16], row-major 4x4 mapping
 *                  sweep s into the current frame (Eq. 6).
 *   rois           device, mmbev_roi_t [num_rois], most critical first.
 *   num_rois       0 <= num_rois <= MMBEV_MAX_ROIS_PER_FRAME; 0 gives no voxels.
 *   roi_margin     r of Eq. 1, >= 0 and finite, metres.
 *   voxel_size     host, float [3], > 0.
 *   range          host, float [6] (xmin, ymin, zmin, xmax, ymax, zmax), max > min;
 *                  nx*ny*nz must stay below 2^32.
 *   max_pts_per_voxel  K, 1 <= K <= MMBEV_MAX_PTS_PER_VOXEL.
 *   max_voxels     >= 0.
 *   out_feats      device, float32 [max_voxels][5]
 *   out_coords     device, int32 [max_voxels][3] as (z, y, x)
 *   out_counts     device, int32 [max_voxels], min(points in voxel, K)
 *   out_nvox       device, int32 scalar, min(voxels, max_voxels)
 * Rows at and beyond *out_nvox are left untouched.
 */
int mmbev_voxelize_roi(const float *points, const int64_t *sweep_offsets,
                       int32_t num_sweeps, const float *sweep_tf,
                       const mmbev_roi_t *rois, int32_t num_rois, float roi_margin,
                       const float voxel_size[3], const float range[6],
                       int32_t max_pts_per_voxel, int32_t max_voxels,
                       float *out_feats, int32_t *out_coords, int32_t *out_counts,
                       int32_t *out_nvox, void *workspace, size_t workspace_bytes,
                       cudaStream_t stream);

/*
 * num_frames independent frames in one call; the result equals num_frames
 * separate mmbev_voxelize_roi calls.
 *   frame_sweep_offsets  host, int32 [num_frames+1]: frame f owns sweeps
 *                        [fso[f], fso[f+1]); fso[0] = 0, fso[F] = num_sweeps.
 *   frame_roi_offsets    host, int32 [num_frames+1]: frame f owns ROIs
 *                        [fro[f], fro[f+1]) (its own criticality order);
 *                        fro[0] = 0, fro[F] = num_rois.
 *   Outputs are per frame with a stride of max_voxels rows: frame f's voxel v
 *   is row f*max_voxels + v; out_nvox is int32 [num_frames].
 * Other arguments as for mmbev_voxelize_roi; num_rois counts all frames.
 */
int mmbev_voxelize_roi_batched(const float *points, const int64_t *sweep_offsets,
                               int32_t num_sweeps, const float *sweep_tf,
                               const mmbev_roi_t *rois, int32_t num_rois,
                               float roi_margin, const float voxel_size[3],
                               const float range[6], int32_t max_pts_per_voxel,
                               int32_t max_voxels, int32_t num_frames,
                               const int32_t *frame_sweep_offsets,
                               const int32_t *frame_roi_offsets,
                               float *out_feats, int32_t *out_coords,
                               int32_t *out_counts, int32_t *out_nvox,
                               void *workspace, size_t workspace_bytes,
                               cudaStream_t stream);

/*
 * Steps S1-S2 alone, per point (Eq. 6; Alg. 1 inside-ROI test; voxel index),
 * for the same inputs as mmbev_voxelize_roi_batched:
 *   out_xyz   device, float32 [N][3], compensated coordinates of every point
 *   out_lin   device, int64 [N], frame-local voxel linear index, -1 if dropped
 *   out_rank  device, int32 [N], ROI rank, -1 if dropped
 * Needs only the workspace.
 */
int mmbev_classify_points(const float *points, const int64_t *sweep_offsets,
                          int32_t num_sweeps, const float *sweep_tf,
                          const mmbev_roi_t *rois, int32_t num_rois, float roi_margin,
                          const float voxel_size[3], const float range[6],
                          int32_t num_frames, const int32_t *frame_sweep_offsets,
                          const int32_t *frame_roi_offsets, float *out_xyz,
                          int64_t *out_lin, int32_t *out_rank,
                          void *workspace, size_t workspace_bytes, cudaStream_t stream);

/*
 * The prepared form of ROI boxes that the inside test of Alg. 1 uses (Eq. 1
 * box with its margin; Sec. IV-F), as the voxelize calls compute it on the
 * device, for checking against an independent evaluation:
 *   rois        device, mmbev_roi_t [num_rois].
 *   roi_margin  r of Eq. 1, >= 0 and finite.
 *   out         device, float32 [num_rois][6]: cx, cy, c = (float)cos((double)yaw),
 *               s = (float)sin((double)yaw), hl = 0.5f*l + r, hw = 0.5f*w + r.
 * Asynchronous on `stream`; one kernel.
 */
int mmbev_prep_rois(const mmbev_roi_t *rois, int32_t num_rois, float roi_margin, float *out,
                    cudaStream_t stream);

/*
 * Copy the device status word of the last call that used `workspace` into
 * *host_status (0 = no device-side error, else MMBEV_DEV_* bits). This call
 * synchronizes `stream`.
 */
int mmbev_get_status(const void *workspace, size_t workspace_bytes,
                     uint32_t *host_status, cudaStream_t stream);

/*
 * Execution options for mmbev_voxelize_roi_batched_ex.
 *   stage_events      NULL, or MMBEV_NUM_STAGES+1 events created by the
 *                     caller: event k is recorded on `stream` before stage k
 *                     and the last one after the final stage, so the caller
 *                     can time each kernel with cudaEventElapsedTime.
 *   inject_status     0 for use. A test hook: MMBEV_DEV_* bits that the
 *                     call's first kernel sets in the device status word as
 *                     a device-side failure would (in the first chunk only,
 *                     for mmbev_voxelize_roi_batched_host), so that callers
 *                     can check how a failure is reported without one.
 *   rho_out           keep probability, in [0, 1], of an in-range point inside
 *                     no ROI (Alg. 1; the other entry points use 0). The draw
 *                     for the j-th point of a frame (0-based, within that
 *                     frame) is the (j+1)-th output of SplitMix64 (Steele,
 *                     Lea and Flood, OOPSLA 2014) seeded with `seed`; the
 *                     point is kept when the output's top 24 bits are below
 *                     floor(rho_out * 2^24). A kept background point has rank
 *                     R_f (the frame's ROI count), below every ROI, so the
 *                     voxel cap drops background-only voxels first.
 *                     Outside [0, 1] or NaN: MMBEV_EINVAL.
 *   seed              the generator's seed.
 * The stages, in launch order (mmbev_stage_name): prep, classify, compact,
 * sort (one launch per 9-bit digit of the largest linear index: three on a
 * 1440 x 1440 x 40 grid), runs, emit. An event pair brackets each stage,
 * so the sort's launches are timed together.
 */
#define MMBEV_NUM_STAGES 6
typedef struct mmbev_exec_opts {
    cudaEvent_t *stage_events;
    uint32_t inject_status;
    float rho_out;
    uint64_t seed;
} mmbev_exec_opts_t;

/*
 * The batched call with its inputs in host memory (pinned, for the copies
 * to overlap): frames go up in chunks of chunk_frames on copy_stream, and
 * each chunk is voxelized on `stream` as soon as its copy has landed, so the
 * transfers of later chunks overlap the work on earlier ones. The results
 * are those of mmbev_voxelize_roi_batched_ex on the same inputs (frames are
 * independent; the draws of opts->rho_out use frame-local indices).
 *   h_points, h_sweep_tf, h_rois  host, as points, sweep_tf, rois above.
 *   d_points, d_sweep_tf, d_rois  device staging of the same sizes, written
 *               by the call.
 *   sweep_offsets, frame_*_offsets  host, as above; checked before any copy.
 *   pack_dst, pack_bytes  NULL, or device or pinned host memory of at least
 *               mmbev_pack_size(F, max_voxels) bytes: each chunk's kept rows
 *               are packed there (mmbev_pack_voxels' layout) as soon as the
 *               chunk is done, so the results cross to the host while later
 *               chunks go up and run.
 *   chunk_frames  frames a chunk (>= 1).
 *   copy_stream  the stream of the copies (the call's own `stream` makes it
 *               serial).
 * Everything else as mmbev_voxelize_roi_batched_ex; opts->stage_events must
 * be NULL. The workspace status accumulates over the chunks.
 * Ordering: the call is asynchronous. The host inputs must stay unchanged
 * until the copies have run. The copies are ordered after earlier work on
 * copy_stream only, not on `stream`: a caller that reuses the staging
 * buffers makes copy_stream wait (an event) for the last call that read
 * them. With two staging sets used in turn, a call's uploads overlap the
 * previous call's work (the Python binding does this).
 */
int mmbev_voxelize_roi_batched_host(
    const float *h_points, const int64_t *sweep_offsets, int32_t num_sweeps,
    const float *h_sweep_tf, const mmbev_roi_t *h_rois, int32_t num_rois, float roi_margin,
    const float voxel_size[3], const float range[6], int32_t max_pts_per_voxel,
    int32_t max_voxels, int32_t num_frames, const int32_t *frame_sweep_offsets,
    const int32_t *frame_roi_offsets, float *d_points, float *d_sweep_tf, mmbev_roi_t *d_rois,
    float *out_feats, int32_t *out_coords, int32_t *out_counts, int32_t *out_nvox,
    void *workspace, size_t workspace_bytes, void *pack_dst,
    size_t pack_bytes, int32_t chunk_frames, cudaStream_t stream, cudaStream_t copy_stream,
    const mmbev_exec_opts_t *opts);

int mmbev_voxelize_roi_batched_ex(const float *points, const int64_t *sweep_offsets,
                                  int32_t num_sweeps, const float *sweep_tf,
                                  const mmbev_roi_t *rois, int32_t num_rois,
                                  float roi_margin, const float voxel_size[3],
                                  const float range[6], int32_t max_pts_per_voxel,
                                  int32_t max_voxels, int32_t num_frames,
                                  const int32_t *frame_sweep_offsets,
                                  const int32_t *frame_roi_offsets,
                                  float *out_feats, int32_t *out_coords,
                                  int32_t *out_counts, int32_t *out_nvox,
                                  void *workspace, size_t workspace_bytes,
                                  cudaStream_t stream, const mmbev_exec_opts_t *opts);

/*
 * Single-frame voxelization for callers that cannot allocate device memory.
 * The paper has no counterpart: this is a deployment variant of
 * mmbev_voxelize_roi. Some callers cannot call cudaMalloc at all, for
 * example a real-time perception process that forbids allocation after
 * start-up (allocation may synchronize the device and has unbounded
 * latency), or a host that owns every device buffer and lends the library
 * only its inputs and outputs. Here the workspace is one file-scope
 * device array of MMBEV_NOALLOC_SCRATCH_BYTES, which every GPU that loads
 * the library keeps until the process exits; the call allocates nothing.
 *   Arguments are those of mmbev_voxelize_roi without the workspace, plus
 *   out_status  device, uint32 scalar or NULL: receives the call's device
 *               status word (MMBEV_DEV_* bits, 0 = no device-side error).
 *   Returns MMBEV_EWORKSPACE, before any launch, when the call needs more
 *   than the array holds: mmbev_workspace_size(N, num_rois, max_voxels, 1,
 *   voxel_size, range) must not exceed MMBEV_NOALLOC_SCRATCH_BYTES; K and
 *   max_voxels do not enter it. On the grids of the tiny, nuScenes- and
 *   Ouster-shaped workloads, with their ROI counts, that allows up to about
 *   1,500,000 points.
 * The first call on a device (and the first in each new context of it, as
 * after cudaDeviceReset) looks up the array's device address with that
 * device current; make that first call before any stream capture. The
 * array keeps the previous call's contents; nothing in it needs to start at
 * zero, since every call initialises the part it reads. All calls on a
 * device share the one array: calls whose executions overlap on the GPU
 * race and must be serialized.
 */
#define MMBEV_NOALLOC_SCRATCH_BYTES (96u << 20)
int mmbev_voxelize_roi_noalloc(const float *points, const int64_t *sweep_offsets,
                               int32_t num_sweeps, const float *sweep_tf,
                               const mmbev_roi_t *rois, int32_t num_rois, float roi_margin,
                               const float voxel_size[3], const float range[6],
                               int32_t max_pts_per_voxel, int32_t max_voxels,
                               float *out_feats, int32_t *out_coords, int32_t *out_counts,
                               int32_t *out_nvox, uint32_t *out_status, cudaStream_t stream);

/* Names of the stages timed by stage_events, for reports. */
const char *mmbev_stage_name(int32_t stage);

/* Library version string. */
const char *mmbev_version(void);

/*
 * Temporal ROIs and criticality ranking (Sec. IV-C; Eq. 1, 3-5, 8): the ROI
 * table a voxelize call takes, built on the device from the previous frame's
 * detections.
 *   objects     device, per frame its detections in the current ego frame
 *               (x forward, y left, metres): box (cx, cy, w, l, yaw), ground
 *               velocity (vx, vy) in m/s along the ego axes, class
 *               MMBEV_CLS_*. Frame f owns objects [off[f], off[f+1]),
 *               at most MMBEV_MAX_ROIS_PER_FRAME / 2 of them.
 *   frame_obj_offsets  host, [num_frames + 1], off[0] = 0, nondecreasing.
 *   params      host: ego speed v_ego along +x, dt of Eq. 1, a_brake and
 *               d_min of Eq. 4, the cone half-angle theta (theta_max_deg at
 *               or below v_wide, theta_min_deg at or above v_narrow, linear
 *               in between; the paper bounds it by 60 and 15 degrees), the
 *               TTC thresholds tau of Eq. 5 for vulnerable and motorized
 *               classes (static objects are geometry-critical only), and
 *               r_coll of Eq. 8. The paper leaves a_brake, d_min, the theta
 *               breakpoints and r_coll open.
 *   out_rois    device, [2 * off[num_frames]]: frame f's ROIs at
 *               [2*off[f], 2*off[f+1]) in rank order, so 2*off serves as
 *               the voxelize call's frame_roi_offsets. Each object gives two
 *               ROIs, its box and its box moved by the relative velocity
 *               (vx - v_ego, vy) times dt (Eq. 1's b and b + v dt).
 *   out_flags   device [off[num_frames]] or NULL: per object (input order)
 *               bit 0 Geom, bit 1 Safety.
 * Ranking: mandatory objects (Geom or Safety) first, then ascending TTC,
 * then ascending squared distance, then input index. Geom: x >= 0,
 * x^2 + y^2 <= dmax^2, |y| <= x * tan(theta), dmax = max(d_min, v_ego^2 /
 * (2 a_brake)) and tan(theta) evaluated in double then rounded to fp32.
 * TTC: relative velocity v = (vx - v_ego, vy); t* = -(p.v)/|v|^2; TTC = t*
 * when t* > 0 and |p + t* v|^2 <= r_coll^2, else infinity. All other
 * arithmetic is fp32, every product and sum rounded in the order written.
 */
#define MMBEV_CLS_MOTOR 0
#define MMBEV_CLS_VRU 1
#define MMBEV_CLS_STATIC 2
typedef struct { float cx, cy, w, l, yaw, vx, vy; int32_t cls; } mmbev_object_t;
typedef struct {
    float v_ego, dt, a_brake, d_min, theta_max_deg, theta_min_deg, v_wide, v_narrow;
    float tau_vru, tau_motor, r_coll;
} mmbev_crit_params_t;

int mmbev_build_rois(const mmbev_object_t *objects, const int32_t *frame_obj_offsets,
                     int32_t num_frames, const mmbev_crit_params_t *params,
                     mmbev_roi_t *out_rois, int32_t *out_flags, cudaStream_t stream);

/*
 * Voxel-grid connected components (the object-cluster proposer of the
 * paper's robot deployment, Sec. VI-F): the kept voxels of each frame joined under
 * 26-connectivity (voxels sharing a face, an edge or a corner).
 *   coords, nvox  device, a voxelize call's outputs ([F*max_voxels][3] (z, y,
 *               x) int32, [F] int32); rows >= nvox[f] are ignored. A frame's
 *               rows must ascend by linear index (as voxelize writes them;
 *               else MMBEV_DEV_UNSORTED is set and the labels are undefined).
 *   dims        host (nx, ny, nz).
 *   table, table_bytes  only when max_voxels > 262,144 (else ignored, may
 *               be NULL): the caller's all-zero device buffer, 16-byte
 *               aligned, of at least mmbev_components_table_size(F,
 *               max_voxels) bytes (else MMBEV_EWORKSPACE): per frame a hash
 *               region of 8-byte slots, then 4 bytes of scratch per row. All
 *               zero again when the work completes.
 *   out_labels  device int32 [F*max_voxels]: for each kept row, the row
 *               (within its frame) of its component's root, the smallest
 *               row of the component; -1 for rows >= nvox[f] and rows whose
 *               coordinates lie outside the grid.
 *   out_comp    device int32 [F*max_voxels][7] or NULL: at each root row the
 *               component's voxel count and bounding box (zmin, ymin, xmin,
 *               zmax, ymax, xmax); other rows are unspecified.
 *   out_ncomp   device int32 [F]: components per frame.
 *   out_status  device uint32 or NULL: MMBEV_DEV_* bits, reset by the call.
 * mmbev_components_table_size returns that table size: 0 when no table is
 * needed, and for sizes out of range; max_voxels <= 2^28. With max_voxels <=
 * 262,144 the work is one launch of one thread-block cluster per frame (the
 * frame's union-find in the cluster's shared memory, neighbours found by
 * the rows' order), else five launches over a frame grid.
 * Asynchronous on `stream`.
 */
size_t mmbev_components_table_size(int32_t num_frames, int32_t max_voxels);
int mmbev_voxel_components(const int32_t *coords, const int32_t *nvox, int32_t num_frames,
                           int32_t max_voxels, const int32_t dims[3], void *table,
                           size_t table_bytes, int32_t *out_labels, int32_t *out_comp,
                           int32_t *out_ncomp, uint32_t *out_status, cudaStream_t stream);

/*
 * Packing of a voxelize call's outputs for the host: every frame's kept rows
 * [0, nvox[f]) gathered, frame after frame, into one contiguous buffer, so
 * the result crosses to the host in one transfer (or, with dst in pinned
 * host memory, is written there by the device directly).
 *   feats, coords, counts, nvox  device, a voxelize call's outputs (frame f's
 *               rows start at f*max_voxels).
 *   dst, dst_bytes  device memory or pinned host memory, 4-byte aligned, at
 *               least mmbev_pack_size(F, max_voxels) bytes (else
 *               MMBEV_EWORKSPACE): int32 off[F+1] (off[f] = the first record
 *               of frame f, off[F] = the total T), then T records of nine
 *               4-byte words: the five fp32 means, then z, y, x and the point
 *               count as int32.
 * Asynchronous on `stream`; one kernel.
 */
size_t mmbev_pack_size(int32_t num_frames, int32_t max_voxels);
int mmbev_pack_voxels(const float *feats, const int32_t *coords, const int32_t *counts,
                      const int32_t *nvox, int32_t num_frames, int32_t max_voxels, void *dst,
                      size_t dst_bytes, cudaStream_t stream);

/*
 * ScatterToBEV (Alg. 1, last step): the voxel features of F frames written
 * into a dense, zero-initialized canvas by voxel coordinate.
 *   feats, coords, nvox  device, the outputs of a voxelize call: feats
 *               [F*max_voxels][5] fp32, coords [F*max_voxels][3] int32
 *               (z, y, x), nvox [F] int32; frame f's rows start at
 *               f*max_voxels and rows >= nvox[f] are ignored.
 *   dims        host, the grid (nx, ny, nz), each >= 1.
 *   canvas      device fp32 [F][nz*5][ny][nx]: channel cz*5 + c of cell
 *               (cy, cx) holds feature c of voxel (cz, cy, cx); for a pillar
 *               grid (nz = 1) that is the usual [5][ny][nx] BEV map. The call
 *               zero-fills it first. canvas_bytes must be at least
 *               F*nz*5*ny*nx*4 (else MMBEV_EWORKSPACE) and the canvas 16-byte
 *               aligned (else MMBEV_EINVAL).
 * Voxels whose coordinates lie outside dims are skipped. Asynchronous on
 * `stream`; the library owns no memory.
 */
int mmbev_scatter_bev(const float *feats, const int32_t *coords, const int32_t *nvox,
                      int32_t num_frames, int32_t max_voxels, const int32_t dims[3],
                      float *canvas, size_t canvas_bytes, cudaStream_t stream);

/*
 * ScatterToBEV for a stream of calls: a canvas that holds exactly the
 * scatter of the previous outputs (prev_coords, prev_nvox: device, the same
 * shapes as coords, nvox; both NULL for an all-zero canvas) gets the cells of
 * those voxels zeroed, then the new voxels written. The canvas equals the
 * one mmbev_scatter_bev gives for (feats, coords, nvox), without the fill of
 * the whole canvas. prev and the new outputs must not alias. Other arguments
 * and errors as mmbev_scatter_bev.
 */
int mmbev_scatter_bev_update(const int32_t *prev_coords, const int32_t *prev_nvox,
                             const float *feats, const int32_t *coords, const int32_t *nvox,
                             int32_t num_frames, int32_t max_voxels, const int32_t dims[3],
                             float *canvas, size_t canvas_bytes, cudaStream_t stream);

#ifdef __cplusplus
}
#endif

#endif /* MMBEV_H_ */
