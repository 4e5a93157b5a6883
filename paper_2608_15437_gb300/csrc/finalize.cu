// Stage 8: voxel feature encoder (S5 of the path; Alg. 1 "VoxelFeatureEncoder").
//
// One thread per kept voxel, in output order. The voxel's slot holds the
// bitwise-NOT of its K smallest point indices, largest first, i.e. in
// ascending point index. The thread gathers those points, recomputes their
// motion-compensated coordinates with the same fp32 operation order as the
// point pass (Eq. 6), sums (x', y', z', intensity, dt) in index order, divides
// once by the count, writes the feature row and the count, and returns the
// slot to the all-zero state.
#include "mmbev_internal.cuh"

namespace mmbev {
namespace {

constexpr int kThreads = 256;

__global__ void __launch_bounds__(kThreads) k_finalize(Params p) {
    __shared__ uint32_t s_vbase[kMaxFrames + 1];
    __shared__ int64_t s_soff[kMaxSweeps + 1];
    const int F = p.num_frames, S = p.num_sweeps;
    for (int i = threadIdx.x; i < F; i += blockDim.x) s_vbase[i] = p.finfo[i].vbase;
    for (int i = threadIdx.x; i <= S; i += blockDim.x) s_soff[i] = p.sweep_off[i];
    const uint32_t total = ld_cg(&p.hdr->total_kept);
    if (threadIdx.x == 0) s_vbase[F] = total;
    __syncthreads();
    const uint32_t gs = gridDim.x * blockDim.x;
    const int K = p.K;
    for (uint32_t g = blockIdx.x * blockDim.x + threadIdx.x; g < total; g += gs) {
        int lo = 0, hi = F;  // s_vbase[lo] <= g < s_vbase[hi]
        while (hi - lo > 1) {
            const int mid = (lo + hi) >> 1;
            if (s_vbase[mid] <= g) lo = mid; else hi = mid;
        }
        const int f = lo;
        const uint32_t vid = g - s_vbase[f];
        const uint32_t h = p.vid_slot[g];
        const uint32_t* tk = slot_topk(p, h);
        float acc[5] = {0.f, 0.f, 0.f, 0.f, 0.f};
        int cnt = 0;
        int s = 0;
        for (int j0 = 0; j0 < K; j0 += 4) {
            const uint4 q = __ldcg(reinterpret_cast<const uint4*>(tk + j0));
            const uint32_t lv[4] = {q.x, q.y, q.z, q.w};
            bool done = false;
#pragma unroll
            for (int c = 0; c < 4; ++c) {
                if (j0 + c >= K || lv[c] == 0u) { done = true; break; }
                const int64_t idx = (int64_t)(uint32_t)~lv[c];
                // sweep of idx: indices ascend, so search forward from the last one
                if (cnt == 0) {
                    int a = 0, bnd = S;
                    while (bnd - a > 1) {
                        const int mid = (a + bnd) >> 1;
                        if (s_soff[mid] <= idx) a = mid; else bnd = mid;
                    }
                    s = a;
                } else {
                    while (s + 1 < S && s_soff[s + 1] <= idx) ++s;
                }
                float T[12];
#pragma unroll
                for (int e = 0; e < 12; ++e) T[e] = __ldg(p.sweep_tf + (size_t)s * 16 + e);
                const float* pt = p.points + idx * 5;
                const float px = __ldg(pt + 0), py = __ldg(pt + 1), pz = __ldg(pt + 2);
                const float pi = __ldg(pt + 3), pd = __ldg(pt + 4);
                float x, y, z;
                compensate(T, px, py, pz, x, y, z);
                acc[0] = __fadd_rn(acc[0], x);
                acc[1] = __fadd_rn(acc[1], y);
                acc[2] = __fadd_rn(acc[2], z);
                acc[3] = __fadd_rn(acc[3], pi);
                acc[4] = __fadd_rn(acc[4], pd);
                ++cnt;
            }
            if (done) break;
        }
        const size_t row = (size_t)f * (uint32_t)p.max_voxels + vid;
        const float fc = (float)cnt;
#pragma unroll
        for (int c = 0; c < 5; ++c) p.out_feats[row * 5 + c] = __fdiv_rn(acc[c], fc);
        p.out_counts[row] = cnt;
        // release the slot
        uint4* sl = reinterpret_cast<uint4*>(p.table + (size_t)h * p.slot_stride);
        const uint32_t n16 = p.slot_stride / 16;
        for (uint32_t i = 0; i < n16; ++i) sl[i] = make_uint4(0u, 0u, 0u, 0u);
    }
}

}  // namespace

cudaError_t launch_finalize(const Params& p, int num_sms, cudaStream_t st) {
    k_finalize<<<num_sms * 4, kThreads, 0, st>>>(p);
    return cudaGetLastError();
}

}  // namespace mmbev
