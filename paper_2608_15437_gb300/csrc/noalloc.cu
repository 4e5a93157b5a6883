// mmbev_voxelize_roi_noalloc: the single-frame call for callers that cannot
// allocate device memory.
//
// Some callers cannot call cudaMalloc at all: a real-time perception process
// that forbids allocation after start-up (allocation can synchronize the
// device and has unbounded latency), a host that hands the library only
// pre-registered input and output buffers, or code running where the CUDA
// allocator is owned by another framework. This entry point serves them: the
// hash table and the scratch workspace live in one file-scope device array of
// MMBEV_NOALLOC_SCRATCH_BYTES, which every GPU that loads this library holds
// until the process exits. The caller passes only inputs and outputs.
//
// The array is shared by every call on a device and keeps the last call's
// contents, so each call first zeroes the part that must start at zero (the
// hash table). Calls whose executions overlap on the GPU (two streams, or two
// host threads) race on the array; serialize them.
#include <atomic>
#include <cstring>

#include "mmbev_internal.cuh"

namespace {

// Scratch of the no-allocation entry point: the hash table, then the workspace.
static __device__ __align__(256) unsigned char g_noalloc_scratch[MMBEV_NOALLOC_SCRATCH_BYTES];

constexpr int kMaxDevices = 64;
std::atomic<void*> g_scratch_addr[kMaxDevices];

size_t round256(size_t x) { return (x + 255) / 256 * 256; }

// Device address of g_noalloc_scratch on the current device. In host code
// the array's name is only a stand-in, so the address is looked up once per
// device with that device current, on the first call.
cudaError_t scratch_address(void** out) {
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    if (dev < 0 || dev >= kMaxDevices) return cudaErrorInvalidDevice;
    void* p = g_scratch_addr[dev].load(std::memory_order_acquire);
    if (p == nullptr) {
        e = cudaGetSymbolAddress(&p, g_noalloc_scratch);
        if (e != cudaSuccess) return e;
        g_scratch_addr[dev].store(p, std::memory_order_release);
    }
    *out = p;
    return cudaSuccess;
}

}  // namespace

extern "C" int mmbev_voxelize_roi_noalloc(const float* points, const int64_t* sweep_offsets,
                                          int32_t num_sweeps, const float* sweep_tf,
                                          const mmbev_roi_t* rois, int32_t num_rois,
                                          float roi_margin, const float voxel_size[3],
                                          const float range[6], int32_t max_pts_per_voxel,
                                          int32_t max_voxels, float* out_feats,
                                          int32_t* out_coords, int32_t* out_counts,
                                          int32_t* out_nvox, uint32_t* out_status,
                                          cudaStream_t stream) {
    if (!sweep_offsets || num_sweeps < 0 || num_sweeps > MMBEV_MAX_SWEEPS) return MMBEV_EINVAL;
    const int64_t n = sweep_offsets[num_sweeps];
    if (n < 0) return MMBEV_EINVAL;
    const size_t table_bytes = mmbev_table_size(n, max_pts_per_voxel);
    const size_t ws_bytes = mmbev_workspace_size(n, num_rois, max_voxels, 1, voxel_size, range);
    if (table_bytes == 0 || ws_bytes == 0) return MMBEV_EINVAL;
    const size_t ws_off = round256(table_bytes);
    if (ws_off + ws_bytes > (size_t)MMBEV_NOALLOC_SCRATCH_BYTES) return MMBEV_EWORKSPACE;

    void* base = nullptr;
    if (scratch_address(&base) != cudaSuccess) return MMBEV_ECUDA;
    unsigned char* scratch = static_cast<unsigned char*>(base);
    // The previous call may have left anything here: zero the table region.
    if (mmbev::launch_zero(scratch, table_bytes, stream) != cudaSuccess) return MMBEV_ECUDA;
    const int rc = mmbev_voxelize_roi(points, sweep_offsets, num_sweeps, sweep_tf, rois, num_rois,
                                      roi_margin, voxel_size, range, max_pts_per_voxel,
                                      max_voxels, out_feats, out_coords, out_counts, out_nvox,
                                      scratch, table_bytes, scratch + ws_off, ws_bytes, stream);
    if (rc != MMBEV_OK) return rc;
    if (out_status) {
        // the device status word is the first word of the workspace
        if (cudaMemcpyAsync(out_status, scratch + ws_off, sizeof(uint32_t),
                            cudaMemcpyDeviceToDevice, stream) != cudaSuccess)
            return MMBEV_ECUDA;
    }
    return MMBEV_OK;
}
