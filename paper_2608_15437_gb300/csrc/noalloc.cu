// mmbev_voxelize_roi_noalloc: the single-frame call for callers that cannot
// allocate device memory.
//
// Some callers cannot call cudaMalloc at all: a real-time perception process
// that forbids allocation after start-up (allocation can synchronize the
// device and has unbounded latency), a host that hands the library only
// pre-registered input and output buffers, or code running where the CUDA
// allocator is owned by another framework. This entry point serves them: the
// scratch workspace lives in one file-scope device array of
// MMBEV_NOALLOC_SCRATCH_BYTES, which every GPU that loads this library holds
// until the process exits. The caller passes only inputs and outputs.
//
// The array is shared by every call on a device and keeps the last call's
// contents. Nothing in it has to start at zero: the call's first kernel
// clears the counters and histograms the later ones accumulate into, and
// each look-back chain's words are cleared by a kernel that runs before the
// one that uses them. Calls whose
// executions overlap on the GPU (two streams, or two host threads) race on
// the array; serialize them.
#include <cuda.h>   // driver types only: the two entry points below are fetched at run time

#include <cstring>
#include <mutex>

#include "mmbev_internal.cuh"

namespace {

// Scratch of the no-allocation entry point: the workspace of its call.
static __device__ __align__(256) unsigned char g_noalloc_scratch[MMBEV_NOALLOC_SCRATCH_BYTES];

constexpr int kMaxDevices = 64;

// Driver calls that name the current context, fetched through the runtime so
// that the library keeps no link-time dependency on the driver library.
using CtxGetCurrentFn = CUresult (*)(CUcontext*);
using CtxGetIdFn = CUresult (*)(CUcontext, unsigned long long*);

struct DriverFns {
    CtxGetCurrentFn get_current = nullptr;
    CtxGetIdFn get_id = nullptr;
    bool ok = false;
};

const DriverFns& driver_fns() {
    static DriverFns fns = [] {
        DriverFns f;
        void* a = nullptr;
        void* b = nullptr;
        cudaDriverEntryPointQueryResult qa = cudaDriverEntryPointSymbolNotFound;
        cudaDriverEntryPointQueryResult qb = cudaDriverEntryPointSymbolNotFound;
        if (cudaGetDriverEntryPointByVersion("cuCtxGetCurrent", &a, 12000, cudaEnableDefault,
                                             &qa) == cudaSuccess &&
            cudaGetDriverEntryPointByVersion("cuCtxGetId", &b, 12000, cudaEnableDefault, &qb) ==
                cudaSuccess &&
            qa == cudaDriverEntryPointSuccess && qb == cudaDriverEntryPointSuccess && a && b) {
            f.get_current = reinterpret_cast<CtxGetCurrentFn>(a);
            f.get_id = reinterpret_cast<CtxGetIdFn>(b);
            f.ok = true;
        }
        return f;
    }();
    return fns;
}

// Unique id (for the life of the process) of the context current on this
// thread, or 0 when none is current or the driver cannot say.
unsigned long long current_context_id() {
    const DriverFns& f = driver_fns();
    if (!f.ok) return 0;
    CUcontext ctx = nullptr;
    if (f.get_current(&ctx) != CUDA_SUCCESS || ctx == nullptr) return 0;
    unsigned long long id = 0;
    if (f.get_id(ctx, &id) != CUDA_SUCCESS) return 0;
    return id;
}

struct ScratchCache {
    unsigned long long ctx_id = 0;   // 0: nothing cached
    void* addr = nullptr;
};
std::mutex g_cache_mu;
ScratchCache g_cache[kMaxDevices];

// Device address of g_noalloc_scratch in the current device's context. In
// host code the array's name is only a stand-in, so the address is looked up
// with cudaGetSymbolAddress, with the device current, and cached per device
// together with the id of the context it belongs to. The first call on a
// device does the lookup (and may load the module), so make it before any
// stream capture. A call in another context of the device, or after
// cudaDeviceReset has replaced the primary context, sees a different id and
// looks the address up again instead of using a stale one.
cudaError_t scratch_address(void** out) {
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    if (dev < 0 || dev >= kMaxDevices) return cudaErrorInvalidDevice;
    std::lock_guard<std::mutex> lock(g_cache_mu);
    const unsigned long long id = current_context_id();
    if (id != 0 && g_cache[dev].ctx_id == id) {
        *out = g_cache[dev].addr;
        return cudaSuccess;
    }
    void* p = nullptr;
    e = cudaGetSymbolAddress(&p, g_noalloc_scratch);   // makes the primary context current if none is
    if (e != cudaSuccess) return e;
    // cache only under a known context id; without one, look up every call
    const unsigned long long id2 = current_context_id();
    g_cache[dev].ctx_id = id2;
    g_cache[dev].addr = id2 != 0 ? p : nullptr;
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
    const size_t ws_bytes = mmbev_workspace_size(n, num_rois, max_voxels, 1, voxel_size, range);
    if (ws_bytes == 0) return MMBEV_EINVAL;
    if (ws_bytes > (size_t)MMBEV_NOALLOC_SCRATCH_BYTES) return MMBEV_EWORKSPACE;

    void* base = nullptr;
    if (scratch_address(&base) != cudaSuccess) return MMBEV_ECUDA;
    unsigned char* scratch = static_cast<unsigned char*>(base);
    const int rc = mmbev_voxelize_roi(points, sweep_offsets, num_sweeps, sweep_tf, rois, num_rois,
                                      roi_margin, voxel_size, range, max_pts_per_voxel,
                                      max_voxels, out_feats, out_coords, out_counts, out_nvox,
                                      scratch, ws_bytes, stream);
    if (rc != MMBEV_OK) return rc;
    if (out_status) {
        // the device status word is the first word of the workspace
        if (cudaMemcpyAsync(out_status, scratch, sizeof(uint32_t), cudaMemcpyDeviceToDevice,
                            stream) != cudaSuccess)
            return MMBEV_ECUDA;
    }
    return MMBEV_OK;
}
