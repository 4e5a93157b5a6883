// ScatterToBEV (Alg. 1, last step): kept voxel features written into a dense,
// zero-initialized BEV canvas by voxel coordinate.
//
// Two kernels on the caller's stream: a grid-stride 16-byte zero fill of the
// canvas (it is mostly zeros: the write bandwidth bounds the call), then one
// thread per (frame, output row) that writes the row's five features at
// canvas[f][cz*5 + c][cy][cx]. The second kernel is a programmatic dependent
// of the first and waits for it before writing.
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

__global__ void __launch_bounds__(kBevThreads)
k_bev_scatter(const float* feats, const int32_t* coords, const int32_t* nvox, int32_t F,
              int32_t max_voxels, int32_t nx, int32_t ny, int32_t nz, float* canvas) {
    pdl_wait();
    const size_t rows = (size_t)F * (size_t)max_voxels;
    const size_t plane = (size_t)ny * nx;
    const size_t gs = (size_t)gridDim.x * blockDim.x;
    for (size_t g = (size_t)blockIdx.x * blockDim.x + threadIdx.x; g < rows; g += gs) {
        const int32_t f = (int32_t)(g / (size_t)max_voxels);
        const int32_t v = (int32_t)(g % (size_t)max_voxels);
        if (v >= __ldg(nvox + f)) continue;
        const int32_t cz = __ldg(coords + 3 * g), cy = __ldg(coords + 3 * g + 1),
                      cx = __ldg(coords + 3 * g + 2);
        if (cz < 0 || cz >= nz || cy < 0 || cy >= ny || cx < 0 || cx >= nx) continue;
        float* base = canvas + (size_t)f * nz * 5 * plane + (size_t)cz * 5 * plane +
                      (size_t)cy * nx + cx;
#pragma unroll
        for (int c = 0; c < 5; ++c) base[(size_t)c * plane] = __ldg(feats + 5 * g + c);
    }
}

}  // namespace
}  // namespace mmbev

using namespace mmbev;

extern "C" int mmbev_scatter_bev(const float* feats, const int32_t* coords, const int32_t* nvox,
                                 int32_t num_frames, int32_t max_voxels, const int32_t dims[3],
                                 float* canvas, size_t canvas_bytes, cudaStream_t stream) {
    if (num_frames < 0 || max_voxels < 0 || !dims) return MMBEV_EINVAL;
    if (dims[0] < 1 || dims[1] < 1 || dims[2] < 1) return MMBEV_EINVAL;
    const unsigned long long cells =
        (unsigned long long)dims[0] * (unsigned long long)dims[1] * (unsigned long long)dims[2];
    const unsigned long long need = (unsigned long long)num_frames * cells * 5ull * 4ull;
    if (need == 0) return MMBEV_OK;
    if (!canvas || (reinterpret_cast<uintptr_t>(canvas) & 15u)) return MMBEV_EINVAL;
    if (canvas_bytes < need) return MMBEV_EWORKSPACE;
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
        e = launch_k(k_bev_scatter, dim3((unsigned)sms * 8), dim3(kBevThreads), 0, stream, true,
                     feats, coords, nvox, num_frames, max_voxels, dims[0], dims[1], dims[2],
                     canvas);
        if (e != cudaSuccess) return MMBEV_ECUDA;
    }
    return MMBEV_OK;
}
