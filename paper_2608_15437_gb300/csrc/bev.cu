// ScatterToBEV (Alg. 1, last step): kept voxel features written into a dense,
// zero-initialized BEV canvas by voxel coordinate.
//
// Two kernels on the caller's stream: a grid-stride 16-byte zero fill of the
// canvas (it is mostly zeros: the write bandwidth bounds the call), then one
// thread per kept row, over a frame grid, that writes the row's five
// features at canvas[f][cz*5 + c][cy][cx]. The second kernel is a
// programmatic dependent of the first and waits for it before writing.
//
// The update entry replaces the fill: a canvas that holds exactly the
// scatter of the previous outputs gets the cells of those outputs zeroed (one
// thread per previous kept row), then the new rows written, which gives the
// same canvas as a fill and a scatter.
#include <algorithm>
#include <cstdint>

#include "mmbev_internal.cuh"

namespace mmbev {
namespace {

constexpr int kBevThreads = 256;

// Zero n16 16-byte words, then the ntail 4-byte words after them.
__global__ void __launch_bounds__(kBevThreads) k_bev_zero(uint4* canvas, size_t n16, int ntail) {
    const size_t gs = (size_t)gridDim.x * blockDim.x;
    const size_t t = (size_t)blockIdx.x * blockDim.x + threadIdx.x;
    for (size_t i = t; i < n16; i += gs) canvas[i] = make_uint4(0u, 0u, 0u, 0u);
    if (t < (size_t)ntail) reinterpret_cast<uint32_t*>(canvas + n16)[t] = 0u;
}

// One thread per kept row of frame blockIdx.y: the row's cell gets its five
// features (kZero: zeros). Rows outside the grid are skipped.
template <bool kZero>
__global__ void __launch_bounds__(kBevThreads)
k_bev_rows(const float* feats, const int32_t* coords, const int32_t* nvox, int32_t max_voxels,
           int32_t nx, int32_t ny, int32_t nz, float* canvas) {
    pdl_wait();
    const int f = blockIdx.y;
    const int nv = min(max(__ldg(nvox + f), 0), max_voxels);
    const size_t plane = (size_t)ny * nx;
    const size_t rows0 = (size_t)f * (size_t)max_voxels;
    for (int v = blockIdx.x * blockDim.x + threadIdx.x; v < nv; v += gridDim.x * blockDim.x) {
        const size_t g = rows0 + (size_t)v;
        const int32_t cz = __ldg(coords + 3 * g), cy = __ldg(coords + 3 * g + 1),
                      cx = __ldg(coords + 3 * g + 2);
        if (cz < 0 || cz >= nz || cy < 0 || cy >= ny || cx < 0 || cx >= nx) continue;
        float* base = canvas + (size_t)f * nz * 5 * plane + (size_t)cz * 5 * plane +
                      (size_t)cy * nx + cx;
#pragma unroll
        for (int c = 0; c < 5; ++c) base[(size_t)c * plane] = kZero ? 0.f : __ldg(feats + 5 * g + c);
    }
}

// A frame grid of about 8 blocks per SM in all, each frame's blocks striding
// over its kept rows.
dim3 bev_rows_grid(int num_frames, int max_voxels, int sms) {
    const long long per = std::max<long long>(
        1, std::min<long long>(((long long)max_voxels + kBevThreads - 1) / kBevThreads,
                               ((long long)sms * 8 + num_frames - 1) / num_frames));
    return dim3((unsigned)per, (unsigned)num_frames);
}

int bev_check(int32_t num_frames, int32_t max_voxels, const int32_t dims[3], const float* canvas,
              size_t canvas_bytes, unsigned long long* need) {
    if (num_frames < 0 || num_frames > 65535 || max_voxels < 0 || !dims) return MMBEV_EINVAL;
    if (dims[0] < 1 || dims[1] < 1 || dims[2] < 1) return MMBEV_EINVAL;
    const unsigned long long cells =
        (unsigned long long)dims[0] * (unsigned long long)dims[1] * (unsigned long long)dims[2];
    *need = (unsigned long long)num_frames * cells * 5ull * 4ull;
    if (*need == 0) return MMBEV_OK;
    if (!canvas || (reinterpret_cast<uintptr_t>(canvas) & 15u)) return MMBEV_EINVAL;
    if (canvas_bytes < *need) return MMBEV_EWORKSPACE;
    return MMBEV_OK;
}

}  // namespace
}  // namespace mmbev

using namespace mmbev;

extern "C" int mmbev_scatter_bev(const float* feats, const int32_t* coords, const int32_t* nvox,
                                 int32_t num_frames, int32_t max_voxels, const int32_t dims[3],
                                 float* canvas, size_t canvas_bytes, cudaStream_t stream) {
    unsigned long long need = 0;
    const int rc = bev_check(num_frames, max_voxels, dims, canvas, canvas_bytes, &need);
    if (rc != MMBEV_OK || need == 0) return rc;
    if (max_voxels > 0 && (!feats || !coords || !nvox)) return MMBEV_EINVAL;
    int dev = 0, sms = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) return MMBEV_ECUDA;
    if (cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess)
        return MMBEV_ECUDA;
    // the canvas holds need bytes, a multiple of 4: whole 16-byte words, then
    // up to three 4-byte words
    const size_t n16 = (size_t)(need / 16);
    const int ntail = (int)((need % 16) / 4);
    cudaError_t e = launch_k(k_bev_zero, dim3((unsigned)sms * 8), dim3(kBevThreads), 0, stream,
                             false, reinterpret_cast<uint4*>(canvas), n16, ntail);
    if (e != cudaSuccess) return MMBEV_ECUDA;
    if (max_voxels > 0 && num_frames > 0) {
        e = launch_k(k_bev_rows<false>, bev_rows_grid(num_frames, max_voxels, sms),
                     dim3(kBevThreads), 0, stream, true, feats, coords, nvox, max_voxels, dims[0],
                     dims[1], dims[2], canvas);
        if (e != cudaSuccess) return MMBEV_ECUDA;
    }
    return MMBEV_OK;
}

extern "C" int mmbev_scatter_bev_update(const int32_t* prev_coords, const int32_t* prev_nvox,
                                        const float* feats, const int32_t* coords,
                                        const int32_t* nvox, int32_t num_frames,
                                        int32_t max_voxels, const int32_t dims[3], float* canvas,
                                        size_t canvas_bytes, cudaStream_t stream) {
    unsigned long long need = 0;
    const int rc = bev_check(num_frames, max_voxels, dims, canvas, canvas_bytes, &need);
    if (rc != MMBEV_OK || need == 0) return rc;
    if (max_voxels > 0 && (!feats || !coords || !nvox)) return MMBEV_EINVAL;
    if ((prev_coords == nullptr) != (prev_nvox == nullptr)) return MMBEV_EINVAL;
    if (max_voxels == 0) return MMBEV_OK;
    int dev = 0, sms = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) return MMBEV_ECUDA;
    if (cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess)
        return MMBEV_ECUDA;
    const dim3 grid = bev_rows_grid(num_frames, max_voxels, sms);
    cudaError_t e = cudaSuccess;
    if (prev_coords)
        e = launch_k(k_bev_rows<true>, grid, dim3(kBevThreads), 0, stream, false,
                     static_cast<const float*>(nullptr), prev_coords, prev_nvox, max_voxels,
                     dims[0], dims[1], dims[2], canvas);
    if (e == cudaSuccess)
        e = launch_k(k_bev_rows<false>, grid, dim3(kBevThreads), 0, stream, prev_coords != nullptr,
                     feats, coords, nvox, max_voxels, dims[0], dims[1], dims[2], canvas);
    return e == cudaSuccess ? MMBEV_OK : MMBEV_ECUDA;
}
