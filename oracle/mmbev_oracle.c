/*
 * Oracle for ROI-aware multi-sweep LiDAR voxelization (MM-BEV, Sec. IV-D and
 * Sec. IV-F).
 *
 * TEST INFRASTRUCTURE. This file is the plain, slow, single-threaded CPU
 * statement of what the GPU path computes. Only the test suite, the smoke
 * check and the benchmark's CPU-baseline leg may load it. It shares no code,
 * header, table or helper with the CUDA library; the two meet only through
 * the seeded input generator.
 *
 * Build: gcc -O2 -ffp-contract=off -fPIC -shared (contraction off so that
 * every fp32 multiply and add is rounded on its own, as the GPU path does).
 *
 * What is computed, step by step, in the order the paper gives it:
 *   1. Eq. 6 / Eq. 7: each point of sweep s is mapped into the current frame
 *      by that sweep's rotation and translation, p' = R p + T, taken from a
 *      row-major 4x4 whose last row is ignored. fp32, each product and sum
 *      rounded, summed left to right: ((r0*x + r1*y) + r2*z) + t.
 *   2. Range crop: xmin <= x' < xmax (same for y, z). NaN fails.
 *   3. Alg. 1 (inside-any-box test) with the boxes of Eq. 1: a point is kept
 *      when it lies inside some ROI box, the box grown by the margin r on each
 *      half-extent. The ROIs arrive in criticality order (Sec. IV-C); the
 *      point's rank is the index of the first box that contains it. A point
 *      inside no box is kept with probability rho_out (Alg. 1), decided by
 *      one draw of a counter-based generator: SplitMix64 (Steele, Lea and
 *      Flood, OOPSLA 2014) seeded with `seed`, its (j+1)-th output for the
 *      frame's j-th point; the point is kept when the top 24 bits of that
 *      output are below floor(rho_out * 2^24). Such a background point has
 *      rank R (the frame's ROI count): below every ROI in criticality.
 *   4. Hard voxelization (Sec. IV-F): voxel c = floor((p' - min) / size) per
 *      axis, dropped when c >= n; linear index lin = (cz*ny + cy)*nx + cx.
 *      Each voxel keeps the K points with the smallest input index. When more
 *      voxels than max_voxels exist, the max_voxels smallest by
 *      (minimum rank, lin) are kept, so mandatory ROIs keep full fidelity
 *      (Sec. IV-C). Output voxels are in ascending lin.
 *   5. Voxel feature encoder (Alg. 1): mean of (x', y', z', intensity, dt)
 *      over the kept points, an fp32 sum in index order and one fp32 divide.
 *
 * Batched form: every frame is an independent problem; frame f owns sweeps
 * [fso[f], fso[f+1]) and ROIs [fro[f], fro[f+1]); its outputs start at row
 * f*max_voxels.
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

typedef struct { float cx, cy, w, l, yaw; } oracle_roi_t;

enum { ORACLE_OK = 0, ORACLE_EINVAL = -1, ORACLE_ENOMEM = -5 };

/* One kept point: voxel linear index, input index, ROI rank, features. */
typedef struct {
    int64_t lin;
    int64_t idx;
    int32_t rank;
    float f[5];
} kept_point_t;

/* One voxel: its linear index, first member in the sorted list, size, and
 * the smallest ROI rank among its points. */
typedef struct {
    int64_t lin;
    int64_t start;
    int64_t n;
    int32_t minrank;
} voxel_t;

/* SplitMix64: the n-th output (n >= 1) of the stream that starts at state
 * `seed` is the finalizer applied to seed + n * 0x9E3779B97F4A7C15. */
static uint64_t splitmix64_nth(uint64_t seed, uint64_t n)
{
    uint64_t z = seed + n * 0x9E3779B97F4A7C15ull;
    z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
    z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
    return z ^ (z >> 31);
}

/* Exposed for the pins: the n-th output of the stream seeded with `seed`. */
uint64_t oracle_splitmix64(uint64_t seed, uint64_t n) { return splitmix64_nth(seed, n); }

/* floor(rho * 2^24) for rho in [0, 1], the keep threshold of a draw's top
 * 24 bits. */
static uint32_t keep_threshold(float rho)
{
    if (!(rho > 0.0f)) return 0u;
    if (rho >= 1.0f) return 1u << 24;
    return (uint32_t)floor((double)rho * 16777216.0);
}

/* Grid extent along one axis: round((max - min) / size) in double. */
static int64_t grid_dim(float lo, float hi, float size)
{
    return (int64_t)llround(((double)hi - (double)lo) / (double)size);
}

/* Eq. 6: rotate and translate one point with the 4x4 T (row-major). */
static void compensate(const float *T, float x, float y, float z,
                       float *xo, float *yo, float *zo)
{
    float a, b, c;
    a = T[0] * x; b = T[1] * y; a = a + b; c = T[2] * z; a = a + c; *xo = a + T[3];
    a = T[4] * x; b = T[5] * y; a = a + b; c = T[6] * z; a = a + c; *yo = a + T[7];
    a = T[8] * x; b = T[9] * y; a = a + b; c = T[10] * z; a = a + c; *zo = a + T[11];
}

/* Eq. 1 box, rotated by yaw, half-extents grown by the margin: the heading's
 * cosine and sine (libm, in double, rounded to fp32) and the two half-extents
 * (l along the heading, w across it). */
static void roi_box(const oracle_roi_t *r, float margin, float out[4])
{
    out[0] = (float)cos((double)r->yaw);
    out[1] = (float)sin((double)r->yaw);
    out[2] = 0.5f * r->l + margin;
    out[3] = 0.5f * r->w + margin;
}

/* Exposed for the pins: roi_box of n ROIs, out[n][4] = (c, s, hl, hw). */
void oracle_roi_boxes(const oracle_roi_t *r, int32_t n, float margin, float *out)
{
    for (int32_t i = 0; i < n; ++i) roi_box(&r[i], margin, out + 4 * (size_t)i);
}

/* The point is inside the box when its coordinates in the box frame lie
 * within the half-extents (boundary included). */
static int inside_roi(const oracle_roi_t *r, float margin, float x, float y)
{
    float box[4];
    roi_box(r, margin, box);
    float c = box[0], s = box[1], hl = box[2], hw = box[3];
    float dx = x - r->cx;
    float dy = y - r->cy;
    float p, q, u, v;
    p = dx * c; q = dy * s; u = p + q;
    p = dy * c; q = dx * s; v = p - q;
    return fabsf(u) <= hl && fabsf(v) <= hw;
}

static int validate_grid(const float vs[3], const float range[6], int64_t dims[3])
{
    for (int a = 0; a < 3; ++a) {
        if (!(vs[a] > 0.0f) || !isfinite(vs[a])) return ORACLE_EINVAL;
        if (!isfinite(range[a]) || !isfinite(range[a + 3])) return ORACLE_EINVAL;
        if (!(range[a + 3] > range[a])) return ORACLE_EINVAL;
        dims[a] = grid_dim(range[a], range[a + 3], vs[a]);
        if (dims[a] < 1) return ORACLE_EINVAL;
    }
    return ORACLE_OK;
}

/*
 * Steps 1-4 for every point, in input order: writes the compensated
 * coordinates, the voxel linear index (-1 when dropped) and the ROI rank
 * (-1 when dropped). The per-point view of the path, used to test the first
 * two steps on their own.
 */
int oracle_classify(const float *points, const int64_t *sweep_offsets,
                    int32_t num_sweeps, const float *sweep_tf,
                    const oracle_roi_t *rois, int32_t num_rois, float margin,
                    const float voxel_size[3], const float range[6],
                    float *out_xyz, int64_t *out_lin, int32_t *out_rank)
{
    int64_t dims[3];
    if (num_sweeps < 0 || num_rois < 0) return ORACLE_EINVAL;
    if (validate_grid(voxel_size, range, dims) != ORACLE_OK) return ORACLE_EINVAL;
    for (int32_t s = 0; s < num_sweeps; ++s) {
        const float *T = sweep_tf + 16 * (int64_t)s;
        for (int64_t i = sweep_offsets[s]; i < sweep_offsets[s + 1]; ++i) {
            const float *p = points + 5 * i;
            float x, y, z;
            compensate(T, p[0], p[1], p[2], &x, &y, &z);
            out_xyz[3 * i + 0] = x;
            out_xyz[3 * i + 1] = y;
            out_xyz[3 * i + 2] = z;
            out_lin[i] = -1;
            out_rank[i] = -1;
            if (!(range[0] <= x && x < range[3])) continue;
            if (!(range[1] <= y && y < range[4])) continue;
            if (!(range[2] <= z && z < range[5])) continue;
            int32_t rank = -1;
            for (int32_t r = 0; r < num_rois; ++r) {
                if (inside_roi(&rois[r], margin, x, y)) { rank = r; break; }
            }
            if (rank < 0) continue;
            int64_t cx = (int64_t)floorf((x - range[0]) / voxel_size[0]);
            int64_t cy = (int64_t)floorf((y - range[1]) / voxel_size[1]);
            int64_t cz = (int64_t)floorf((z - range[2]) / voxel_size[2]);
            if (cx >= dims[0] || cy >= dims[1] || cz >= dims[2]) continue;
            out_lin[i] = (cz * dims[1] + cy) * dims[0] + cx;
            out_rank[i] = rank;
        }
    }
    return ORACLE_OK;
}

static int cmp_point(const void *a, const void *b)
{
    const kept_point_t *p = (const kept_point_t *)a, *q = (const kept_point_t *)b;
    if (p->lin != q->lin) return p->lin < q->lin ? -1 : 1;
    if (p->idx != q->idx) return p->idx < q->idx ? -1 : 1;
    return 0;
}

static int cmp_voxel_rank_lin(const void *a, const void *b)
{
    const voxel_t *u = (const voxel_t *)a, *v = (const voxel_t *)b;
    if (u->minrank != v->minrank) return u->minrank < v->minrank ? -1 : 1;
    if (u->lin != v->lin) return u->lin < v->lin ? -1 : 1;
    return 0;
}

static int cmp_voxel_lin(const void *a, const void *b)
{
    const voxel_t *u = (const voxel_t *)a, *v = (const voxel_t *)b;
    if (u->lin != v->lin) return u->lin < v->lin ? -1 : 1;
    return 0;
}

/* One frame, host pointers. Sweep s of the frame covers points
 * [sweep_offsets[s], sweep_offsets[s+1]); indices are global, so "first K by
 * input index" compares global indices. Rows >= *out_nvox are not written. */
int oracle_voxelize_roi(const float *points, const int64_t *sweep_offsets,
                        int32_t num_sweeps, const float *sweep_tf,
                        const oracle_roi_t *rois, int32_t num_rois, float margin,
                        const float voxel_size[3], const float range[6],
                        int32_t max_pts_per_voxel, int32_t max_voxels,
                        float rho_out, uint64_t seed,
                        float *out_feats, int32_t *out_coords,
                        int32_t *out_counts, int32_t *out_nvox)
{
    int64_t dims[3];
    if (num_sweeps < 0 || num_rois < 0 || max_pts_per_voxel < 1 || max_voxels < 0)
        return ORACLE_EINVAL;
    if (validate_grid(voxel_size, range, dims) != ORACLE_OK) return ORACLE_EINVAL;
    if (!(margin >= 0.0f)) return ORACLE_EINVAL;
    if (!(rho_out >= 0.0f && rho_out <= 1.0f)) return ORACLE_EINVAL;
    const uint32_t thr = keep_threshold(rho_out);

    int64_t first = num_sweeps > 0 ? sweep_offsets[0] : 0;
    int64_t last = num_sweeps > 0 ? sweep_offsets[num_sweeps] : 0;
    int64_t npts = last - first;
    kept_point_t *kept = (kept_point_t *)malloc(sizeof(kept_point_t) * (size_t)(npts > 0 ? npts : 1));
    if (!kept) return ORACLE_ENOMEM;
    int64_t m = 0;

    /* Steps 1-4 (per point). */
    for (int32_t s = 0; s < num_sweeps; ++s) {
        const float *T = sweep_tf + 16 * (int64_t)s;
        for (int64_t i = sweep_offsets[s]; i < sweep_offsets[s + 1]; ++i) {
            const float *p = points + 5 * i;
            float x, y, z;
            compensate(T, p[0], p[1], p[2], &x, &y, &z);
            if (!(range[0] <= x && x < range[3])) continue;
            if (!(range[1] <= y && y < range[4])) continue;
            if (!(range[2] <= z && z < range[5])) continue;
            int32_t rank = -1;
            for (int32_t r = 0; r < num_rois; ++r) {
                if (inside_roi(&rois[r], margin, x, y)) { rank = r; break; }
            }
            if (rank < 0) {
                /* outside every ROI: kept with probability rho_out */
                const uint64_t j = (uint64_t)(i - first);
                if (thr == 0u || (uint32_t)(splitmix64_nth(seed, j + 1) >> 40) >= thr) continue;
                rank = num_rois;
            }
            int64_t cx = (int64_t)floorf((x - range[0]) / voxel_size[0]);
            int64_t cy = (int64_t)floorf((y - range[1]) / voxel_size[1]);
            int64_t cz = (int64_t)floorf((z - range[2]) / voxel_size[2]);
            if (cx >= dims[0] || cy >= dims[1] || cz >= dims[2]) continue;
            kept[m].lin = (cz * dims[1] + cy) * dims[0] + cx;
            kept[m].idx = i;
            kept[m].rank = rank;
            kept[m].f[0] = x;
            kept[m].f[1] = y;
            kept[m].f[2] = z;
            kept[m].f[3] = p[3];
            kept[m].f[4] = p[4];
            ++m;
        }
    }

    /* Group by voxel; inside a voxel, points in input order. */
    qsort(kept, (size_t)m, sizeof(kept_point_t), cmp_point);
    voxel_t *vox = (voxel_t *)malloc(sizeof(voxel_t) * (size_t)(m > 0 ? m : 1));
    if (!vox) { free(kept); return ORACLE_ENOMEM; }
    int64_t u = 0;
    for (int64_t j = 0; j < m; ++j) {
        if (j == 0 || kept[j].lin != kept[j - 1].lin) {
            vox[u].lin = kept[j].lin;
            vox[u].start = j;
            vox[u].n = 0;
            vox[u].minrank = kept[j].rank;
            ++u;
        }
        voxel_t *v = &vox[u - 1];
        v->n += 1;
        if (kept[j].rank < v->minrank) v->minrank = kept[j].rank;
    }

    /* Voxel cap: keep the max_voxels smallest by (minrank, lin), then
     * restore ascending lin. */
    if (u > max_voxels) {
        qsort(vox, (size_t)u, sizeof(voxel_t), cmp_voxel_rank_lin);
        u = max_voxels;
        qsort(vox, (size_t)u, sizeof(voxel_t), cmp_voxel_lin);
    }

    /* Step 5: mean over the first K points of each kept voxel. */
    for (int64_t v = 0; v < u; ++v) {
        int64_t lin = vox[v].lin;
        int64_t cx = lin % dims[0];
        int64_t cy = (lin / dims[0]) % dims[1];
        int64_t cz = lin / (dims[0] * dims[1]);
        int64_t cnt = vox[v].n < max_pts_per_voxel ? vox[v].n : max_pts_per_voxel;
        out_coords[3 * v + 0] = (int32_t)cz;
        out_coords[3 * v + 1] = (int32_t)cy;
        out_coords[3 * v + 2] = (int32_t)cx;
        out_counts[v] = (int32_t)cnt;
        for (int c = 0; c < 5; ++c) {
            float acc = 0.0f;
            for (int64_t j = 0; j < cnt; ++j) acc = acc + kept[vox[v].start + j].f[c];
            out_feats[5 * v + c] = acc / (float)cnt;
        }
    }
    *out_nvox = (int32_t)u;
    free(vox);
    free(kept);
    return ORACLE_OK;
}

/* Batched form: num_frames independent frames, each an oracle_voxelize_roi
 * call on its own sweeps and ROIs (the draws use frame-local point indices,
 * so a batch equals its frames run alone); frame f writes rows starting at
 * f*max_voxels and out_nvox[f]. */
int oracle_voxelize_roi_batched(const float *points, const int64_t *sweep_offsets,
                                int32_t num_sweeps, const float *sweep_tf,
                                const oracle_roi_t *rois, int32_t num_rois,
                                float margin, const float voxel_size[3],
                                const float range[6], int32_t max_pts_per_voxel,
                                int32_t max_voxels, float rho_out, uint64_t seed,
                                int32_t num_frames,
                                const int32_t *frame_sweep_offsets,
                                const int32_t *frame_roi_offsets,
                                float *out_feats, int32_t *out_coords,
                                int32_t *out_counts, int32_t *out_nvox)
{
    if (num_frames < 0) return ORACLE_EINVAL;
    if (num_frames > 0 && (frame_sweep_offsets[num_frames] != num_sweeps ||
                           frame_roi_offsets[num_frames] != num_rois))
        return ORACLE_EINVAL;
    for (int32_t f = 0; f < num_frames; ++f) {
        int32_t s0 = frame_sweep_offsets[f], s1 = frame_sweep_offsets[f + 1];
        int32_t r0 = frame_roi_offsets[f], r1 = frame_roi_offsets[f + 1];
        if (s1 < s0 || r1 < r0) return ORACLE_EINVAL;
        int64_t row = (int64_t)f * max_voxels;
        int rc = oracle_voxelize_roi(points, sweep_offsets + s0, s1 - s0,
                                     sweep_tf + 16 * (int64_t)s0, rois + r0, r1 - r0,
                                     margin, voxel_size, range, max_pts_per_voxel,
                                     max_voxels, rho_out, seed, out_feats + 5 * row,
                                     out_coords + 3 * row, out_counts + row,
                                     out_nvox + f);
        if (rc != ORACLE_OK) return rc;
    }
    return ORACLE_OK;
}

/*
 * Temporal-ROI construction and criticality ranking (Sec. IV-C; Eq. 1, 3-5,
 * 8), one frame. Each object (previous-frame detection, in the current ego
 * frame: x forward, y left) gives two ROIs, its box and the box moved by the
 * relative velocity (vx - v_ego, vy) times dt (Eq. 1's b and b + v dt), in
 * that order. Objects are ranked mandatory first (Geom or Safety), then by
 * TTC, squared distance and input index, all ascending.
 *   Geom (Eq. 3-4): x >= 0, |p|^2 <= dmax^2 and |y| <= x * tan(theta), with
 *     dmax = max(d_min, v_ego^2 / (2 a_brake)) and theta(v_ego) = theta_max
 *     below v_wide, theta_min above v_narrow, linear in between (both in
 *     double, then fp32).
 *   Safety (Eq. 5, 8): class not static and TTC <= tau (VRU or motorized),
 *     TTC = t* = -(p.v)/|v|^2 when t* > 0 and |p + t* v|^2 <= r_coll^2, else
 *     infinity.
 * Arithmetic in fp32, every product and sum rounded, in the order written.
 */
typedef struct { float cx, cy, w, l, yaw, vx, vy; int32_t cls; } oracle_object_t;
typedef struct {
    float v_ego, dt, a_brake, d_min, theta_max_deg, theta_min_deg, v_wide, v_narrow;
    float tau_vru, tau_motor, r_coll;
} oracle_crit_params_t;

typedef struct { int32_t mand; float ttc, d2; int32_t idx; } crit_key_t;

static int cmp_crit(const void *a, const void *b)
{
    const crit_key_t *u = (const crit_key_t *)a, *v = (const crit_key_t *)b;
    if (u->mand != v->mand) return u->mand > v->mand ? -1 : 1;
    if (u->ttc != v->ttc) return u->ttc < v->ttc ? -1 : 1;
    if (u->d2 != v->d2) return u->d2 < v->d2 ? -1 : 1;
    return u->idx < v->idx ? -1 : (u->idx > v->idx);
}

/* The frame-independent thresholds, in double, rounded to fp32. */
void oracle_crit_thresholds(const oracle_crit_params_t *q, float *dmax, float *tan_theta)
{
    const double v = q->v_ego;
    double dm = v * v / (2.0 * (double)q->a_brake);
    if (dm < (double)q->d_min) dm = q->d_min;
    double th;
    if (v <= (double)q->v_wide) th = q->theta_max_deg;
    else if (v >= (double)q->v_narrow) th = q->theta_min_deg;
    else th = (double)q->theta_max_deg +
              ((double)q->theta_min_deg - (double)q->theta_max_deg) * (v - (double)q->v_wide) /
                  ((double)q->v_narrow - (double)q->v_wide);
    *dmax = (float)dm;
    *tan_theta = (float)tan(th * 3.14159265358979323846 / 180.0);
}

int oracle_build_rois(const oracle_object_t *obj, int32_t n, const oracle_crit_params_t *q,
                      oracle_roi_t *out_rois, int32_t *out_flags)
{
    if (n < 0 || !(q->a_brake > 0.0f) || !(q->v_narrow > q->v_wide) || !(q->dt >= 0.0f))
        return ORACLE_EINVAL;
    float dmax, tant;
    oracle_crit_thresholds(q, &dmax, &tant);
    const float dmax2 = dmax * dmax, r2 = q->r_coll * q->r_coll;
    crit_key_t *key = (crit_key_t *)malloc(sizeof(crit_key_t) * (size_t)(n > 0 ? n : 1));
    if (!key) return ORACLE_ENOMEM;
    for (int32_t i = 0; i < n; ++i) {
        const oracle_object_t *o = &obj[i];
        const float px = o->cx, py = o->cy;
        const float rvx = o->vx - q->v_ego, rvy = o->vy;
        float a, b;
        a = px * px; b = py * py; const float d2 = a + b;
        const int geom = px >= 0.0f && d2 <= dmax2 && fabsf(py) <= px * tant;
        float ttc = INFINITY;
        a = rvx * rvx; b = rvy * rvy; const float vv = a + b;
        if (vv > 0.0f) {
            a = px * rvx; b = py * rvy; const float pv = a + b;
            const float t = -pv / vv;
            if (t > 0.0f) {
                a = t * rvx; const float ex = px + a;
                b = t * rvy; const float ey = py + b;
                a = ex * ex; b = ey * ey;
                if (a + b <= r2) ttc = t;
            }
        }
        const float tau = o->cls == 1 ? q->tau_vru : q->tau_motor;
        const int safety = o->cls != 2 && ttc <= tau;
        out_flags[i] = geom | (safety << 1);
        key[i].mand = geom || safety;
        key[i].ttc = ttc;
        key[i].d2 = d2;
        key[i].idx = i;
    }
    qsort(key, (size_t)n, sizeof(crit_key_t), cmp_crit);
    for (int32_t k = 0; k < n; ++k) {
        const oracle_object_t *o = &obj[key[k].idx];
        const float rvx = o->vx - q->v_ego, rvy = o->vy;
        oracle_roi_t r = {o->cx, o->cy, o->w, o->l, o->yaw};
        out_rois[2 * k] = r;
        float m;
        m = rvx * q->dt; r.cx = o->cx + m;
        m = rvy * q->dt; r.cy = o->cy + m;
        out_rois[2 * k + 1] = r;
    }
    free(key);
    return ORACLE_OK;
}
