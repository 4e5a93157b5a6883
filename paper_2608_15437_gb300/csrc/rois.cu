// Temporal ROIs and criticality ranking (Sec. IV-C; Eq. 1, 3-5, 8).
//
// One block per frame. Each thread takes an object: its Geom and Safety
// flags, its time to collision and its squared distance; the block then
// ranks the objects by (mandatory first, TTC, squared distance, index) by
// counting, for every object, the objects with a smaller key, and writes the
// object's two ROIs (its box, and its box moved by the relative velocity
// times dt) at twice its rank. The arithmetic is fp32 with every product and
// sum rounded in a fixed order, so the ranking is exact, not approximate.
#include <cmath>
#include <cstring>

#include "mmbev_internal.cuh"

namespace mmbev {
namespace {

constexpr int kMaxObjects = kMaxRoisPerFrame / 2;

struct CritArgs {
    int32_t off[kMaxFrames + 1];
    float v_ego, dt, dmax2, tan_theta, r2, tau_vru, tau_motor;
};

__global__ void __launch_bounds__(kMaxObjects)
k_build_rois(const mmbev_object_t* obj, const __grid_constant__ CritArgs a, mmbev_roi_t* out,
             int32_t* out_flags) {
    __shared__ int32_t s_mand[kMaxObjects];
    __shared__ float s_ttc[kMaxObjects];
    __shared__ float s_d2[kMaxObjects];
    const int f = blockIdx.x, t = threadIdx.x;
    const int o0 = a.off[f], n = a.off[f + 1] - o0;
    float rvx = 0.f, rvy = 0.f;
    mmbev_object_t o{};
    if (t < n) {
        o = obj[o0 + t];
        const float px = o.cx, py = o.cy;
        rvx = __fsub_rn(o.vx, a.v_ego);
        rvy = o.vy;
        const float d2 = __fadd_rn(__fmul_rn(px, px), __fmul_rn(py, py));
        const bool geom = px >= 0.f && d2 <= a.dmax2 && fabsf(py) <= __fmul_rn(px, a.tan_theta);
        float ttc = INFINITY;
        const float vv = __fadd_rn(__fmul_rn(rvx, rvx), __fmul_rn(rvy, rvy));
        if (vv > 0.f) {
            const float pv = __fadd_rn(__fmul_rn(px, rvx), __fmul_rn(py, rvy));
            const float ts = __fdiv_rn(-pv, vv);
            if (ts > 0.f) {
                const float ex = __fadd_rn(px, __fmul_rn(ts, rvx));
                const float ey = __fadd_rn(py, __fmul_rn(ts, rvy));
                if (__fadd_rn(__fmul_rn(ex, ex), __fmul_rn(ey, ey)) <= a.r2) ttc = ts;
            }
        }
        const float tau = o.cls == MMBEV_CLS_VRU ? a.tau_vru : a.tau_motor;
        const bool safety = o.cls != MMBEV_CLS_STATIC && ttc <= tau;
        if (out_flags) out_flags[o0 + t] = (int32_t)geom | ((int32_t)safety << 1);
        s_mand[t] = geom || safety;
        s_ttc[t] = ttc;
        s_d2[t] = d2;
    }
    __syncthreads();
    if (t >= n) return;
    // rank: objects ahead of this one under (mandatory desc, ttc, d2, index)
    const int m = s_mand[t];
    const float tt = s_ttc[t], dd = s_d2[t];
    int rank = 0;
    for (int j = 0; j < n; ++j) {
        const int mj = s_mand[j];
        const float tj = s_ttc[j], dj = s_d2[j];
        const bool ahead = mj != m ? mj > m
                         : tj != tt ? tj < tt
                         : dj != dd ? dj < dd
                         : j < t;
        rank += ahead;
    }
    mmbev_roi_t r{o.cx, o.cy, o.w, o.l, o.yaw};
    out[2 * (o0 + rank)] = r;
    r.cx = __fadd_rn(o.cx, __fmul_rn(rvx, a.dt));
    r.cy = __fadd_rn(o.cy, __fmul_rn(rvy, a.dt));
    out[2 * (o0 + rank) + 1] = r;
}

}  // namespace
}  // namespace mmbev

using namespace mmbev;

extern "C" int mmbev_build_rois(const mmbev_object_t* objects, const int32_t* frame_obj_offsets,
                                int32_t num_frames, const mmbev_crit_params_t* params,
                                mmbev_roi_t* out_rois, int32_t* out_flags, cudaStream_t stream) {
    if (num_frames < 0 || num_frames > kMaxFrames || !params) return MMBEV_EINVAL;
    if (num_frames > 0 && !frame_obj_offsets) return MMBEV_EINVAL;
    const mmbev_crit_params_t& q = *params;
    const float vals[] = {q.v_ego, q.dt, q.a_brake, q.d_min, q.theta_max_deg, q.theta_min_deg,
                          q.v_wide, q.v_narrow, q.tau_vru, q.tau_motor, q.r_coll};
    for (float v : vals)
        if (!std::isfinite(v)) return MMBEV_EINVAL;
    if (!(q.a_brake > 0.f) || !(q.v_narrow > q.v_wide) || !(q.dt >= 0.f) || !(q.r_coll >= 0.f))
        return MMBEV_EINVAL;
    CritArgs a;
    std::memset(&a, 0, sizeof(a));
    if (num_frames > 0) {
        if (frame_obj_offsets[0] != 0) return MMBEV_EINVAL;
        for (int f = 0; f < num_frames; ++f) {
            const int32_t n = frame_obj_offsets[f + 1] - frame_obj_offsets[f];
            if (n < 0 || n > kMaxObjects) return MMBEV_EINVAL;
        }
        std::memcpy(a.off, frame_obj_offsets, sizeof(int32_t) * (size_t)(num_frames + 1));
    }
    const int32_t total = num_frames > 0 ? frame_obj_offsets[num_frames] : 0;
    if (total > 0 && (!objects || !out_rois)) return MMBEV_EINVAL;
    // the frame-independent thresholds, in double, rounded to fp32 (Eq. 4 and the cone)
    const double v = q.v_ego;
    double dm = v * v / (2.0 * (double)q.a_brake);
    if (dm < (double)q.d_min) dm = q.d_min;
    double th;
    if (v <= q.v_wide) th = q.theta_max_deg;
    else if (v >= q.v_narrow) th = q.theta_min_deg;
    else th = (double)q.theta_max_deg + ((double)q.theta_min_deg - (double)q.theta_max_deg) *
                                            (v - (double)q.v_wide) /
                                            ((double)q.v_narrow - (double)q.v_wide);
    const float dmax = (float)dm;
    a.v_ego = q.v_ego;
    a.dt = q.dt;
    a.dmax2 = dmax * dmax;
    a.tan_theta = (float)std::tan(th * 3.14159265358979323846 / 180.0);
    a.r2 = q.r_coll * q.r_coll;
    a.tau_vru = q.tau_vru;
    a.tau_motor = q.tau_motor;
    if (num_frames == 0 || total == 0) return MMBEV_OK;
    const cudaError_t e = launch_k(k_build_rois, dim3(num_frames), dim3(kMaxObjects), 0, stream,
                                   false, objects, a, out_rois, out_flags);
    return e == cudaSuccess ? MMBEV_OK : MMBEV_ECUDA;
}
