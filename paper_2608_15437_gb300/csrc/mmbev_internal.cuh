// Internal declarations shared by the kernels of libmmbev (sm_103a).
//
// Data layout (one call):
//   points      caller's float32 [N][5] AoS, read once by the point kernel
//               through shared-memory tiles (coalesced 16-byte loads).
//   table       caller's hash table: H = 2^log2 slots of `stride` bytes,
//               slot = { u64 key+1 (0 = empty), u32 0xFFFFFFFF-minrank
//               (0 = none), u32 spare, u32 topk[Kp] }; topk holds the
//               bitwise-NOT of the K smallest point indices of the voxel,
//               kept sorted by a cascade of atomicMax (largest NOT first =
//               smallest index first; 0 = empty level).
//   workspace   Header + per-call arrays (see Layout).
#pragma once

#include <cstdint>
#include <cuda_runtime.h>

#include "mmbev.h"

namespace mmbev {

constexpr int kMaxSweeps = MMBEV_MAX_SWEEPS;
constexpr int kMaxFrames = MMBEV_MAX_FRAMES;
constexpr int kMaxRoisPerFrame = MMBEV_MAX_ROIS_PER_FRAME;
constexpr int kMaxK = MMBEV_MAX_PTS_PER_VOXEL;

// Point kernel tiling: 256 threads, 8 points per thread per tile.
constexpr int kPtsThreads = 256;
constexpr int kPtsPerThread = 8;
constexpr int kTile = kPtsThreads * kPtsPerThread;  // 2048 points = 40 KB

// Bucket bitmap ordering: a bucket spans 2^kBucketLog2 consecutive linear
// indices of one frame; one warp ranks a bucket with two bitmaps in smem.
constexpr int kBucketLog2Max = 13;

// Decoupled look-back scan tile.
constexpr int kScanThreads = 256;
constexpr int kScanPerThread = 8;
constexpr int kScanTile = kScanThreads * kScanPerThread;

// Bounded waits: iterations of a look-back spin before giving up.
constexpr uint32_t kSpinLimit = 1u << 22;

constexpr uint32_t kUnset = 0xFFFFFFFFu;

// Prepared ROI: centre, cos/sin of yaw, half-extents grown by the margin.
struct __align__(16) RoiPrep {
    float cx, cy, c, s;
    float hl, hw, pad0, pad1;
};

// Per-frame results of the cap pass.
struct __align__(16) FrameInfo {
    uint32_t capped;  // more voxels than max_voxels
    uint32_t rstar;   // rank threshold: ranks < rstar kept, == rstar partly
    uint32_t q;       // how many rank-rstar voxels are kept (smallest lin first)
    uint32_t nvox;    // kept voxels
    uint32_t vbase;   // exclusive prefix of nvox over frames
    uint32_t pad[3];
};

// Workspace header; zeroed by the prep kernel at the start of every call.
struct __align__(16) Header {
    uint32_t status;       // MMBEV_DEV_* bits
    uint32_t num_occ;      // occupied slots (unique voxels over all frames)
    uint32_t total_kept;   // kept voxels over all frames
    uint32_t any_capped;   // some frame has more voxels than max_voxels
    uint32_t scan_ticket;  // tile counter of the look-back scan
    uint32_t pad[11];
};

// Everything a kernel needs; passed by value.
struct Params {
    // inputs
    const float* points;
    const float* sweep_tf;
    const mmbev_roi_t* rois;
    int64_t num_points;
    int32_t num_sweeps;
    int32_t num_frames;
    int32_t num_rois;
    int32_t mask_words;     // 32-bit words of ROI bits per coarse cell
    int32_t coarse;         // coarse BEV cells per axis of the candidate mask
    float margin;
    float vs[3];
    float rmin[3];
    float rmax[3];
    float coarse_inv[2];    // coarse cells per metre along x, y
    uint32_t dims[3];       // nx, ny, nz
    uint32_t cells;         // nx*ny*nz
    int32_t K;
    int32_t max_voxels;
    // bucket ordering
    int32_t bucket_log2;
    uint32_t buckets_per_frame;
    uint32_t num_buckets;   // num_frames * buckets_per_frame
    uint32_t scan_tiles;
    // hash table
    uint8_t* table;
    uint32_t table_log2;
    uint32_t slot_stride;   // bytes
    // workspace arrays
    Header* hdr;
    int64_t* sweep_off;     // [S+1]
    int32_t* sweep_frame;   // [S]
    int32_t* frame_sweep_off;  // [F+1]
    int32_t* frame_roi_off;    // [F+1]
    RoiPrep* roi_prep;      // [R]
    uint32_t* masks;        // [F][coarse^2][mask_words]
    uint32_t* hist;         // [R] voxels per minimum rank (capped frames)
    uint32_t* frame_u;      // [F] unique voxels per frame
    FrameInfo* finfo;       // [F]
    unsigned long long* bcnt;  // [B+1] (lo: rank-below count, hi: rank-tie count)
    unsigned long long* scan_agg;  // [tiles]
    unsigned long long* scan_inc;  // [tiles]
    uint32_t* scan_flag;    // [tiles]
    uint32_t* occ;          // [occ_cap] slot of each unique voxel
    uint32_t* d_bucket;     // [occ_cap]
    uint32_t* d_pos;        // [occ_cap] position inside the bucket
    uint32_t* items;        // [occ_cap] voxel ids grouped by bucket
    uint32_t* vid_slot;     // [F*max_voxels] slot of each kept voxel, output order
    uint32_t occ_cap;
    // outputs
    float* out_feats;
    int32_t* out_coords;
    int32_t* out_counts;
    int32_t* out_nvox;
    // classify-only outputs
    float* cls_xyz;
    int64_t* cls_lin;
    int32_t* cls_rank;
};

// Host offsets, copied into the workspace by the prep kernel. Passed by
// value (kernel parameter space), so the host arrays need not outlive the
// call and the call stays capturable in a CUDA graph.
struct HostDesc {
    int64_t sweep_off[kMaxSweeps + 1];
    int32_t frame_sweep_off[kMaxFrames + 1];
    int32_t frame_roi_off[kMaxFrames + 1];
};

// ---------------------------------------------------------------- device helpers

__device__ __forceinline__ void set_status(Header* hdr, uint32_t bits) {
    atomicOr(&hdr->status, bits);
}

// Eq. 6 for one point: ((r0*x + r1*y) + r2*z) + t, every op rounded (no FMA).
__device__ __forceinline__ void compensate(const float* T, float x, float y, float z,
                                           float& xo, float& yo, float& zo) {
    xo = __fadd_rn(__fadd_rn(__fadd_rn(__fmul_rn(T[0], x), __fmul_rn(T[1], y)),
                             __fmul_rn(T[2], z)), T[3]);
    yo = __fadd_rn(__fadd_rn(__fadd_rn(__fmul_rn(T[4], x), __fmul_rn(T[5], y)),
                             __fmul_rn(T[6], z)), T[7]);
    zo = __fadd_rn(__fadd_rn(__fadd_rn(__fmul_rn(T[8], x), __fmul_rn(T[9], y)),
                             __fmul_rn(T[10], z)), T[11]);
}

// Alg. 1 inside test against one prepared ROI (boundary inclusive).
__device__ __forceinline__ bool roi_contains(const RoiPrep& r, float x, float y) {
    const float dx = __fsub_rn(x, r.cx);
    const float dy = __fsub_rn(y, r.cy);
    const float u = __fadd_rn(__fmul_rn(dx, r.c), __fmul_rn(dy, r.s));
    const float v = __fsub_rn(__fmul_rn(dy, r.c), __fmul_rn(dx, r.s));
    return fabsf(u) <= r.hl && fabsf(v) <= r.hw;
}

// Slot addressing.
__device__ __forceinline__ unsigned long long* slot_key(const Params& p, uint32_t h) {
    return reinterpret_cast<unsigned long long*>(p.table + (size_t)h * p.slot_stride);
}
__device__ __forceinline__ uint32_t* slot_rank(const Params& p, uint32_t h) {
    return reinterpret_cast<uint32_t*>(p.table + (size_t)h * p.slot_stride + 8);
}
__device__ __forceinline__ uint32_t* slot_topk(const Params& p, uint32_t h) {
    return reinterpret_cast<uint32_t*>(p.table + (size_t)h * p.slot_stride + 16);
}

// 64-bit mixer (the SplitMix64 finalizer of Steele, Lea and Flood, 2014).
__device__ __forceinline__ uint64_t mix64(uint64_t z) {
    z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
    z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
    return z ^ (z >> 31);
}

// Load at L2 (bypassing the non-coherent L1), for words other blocks update.
__device__ __forceinline__ uint32_t ld_cg(const uint32_t* a) { return __ldcg(a); }
__device__ __forceinline__ unsigned long long ld_cg(const unsigned long long* a) {
    return __ldcg(a);
}

// ---------------------------------------------------------------- launchers

// All launchers enqueue on `st` and return the cudaGetLastError() result.
cudaError_t launch_prep(const Params& p, const HostDesc& d, cudaStream_t st);
cudaError_t launch_points(const Params& p, bool classify_only, cudaStream_t st);
cudaError_t launch_census(const Params& p, int num_sms, cudaStream_t st);
cudaError_t launch_frames(const Params& p, cudaStream_t st);
cudaError_t launch_capped_census(const Params& p, int num_sms, cudaStream_t st);
cudaError_t launch_scan(const Params& p, cudaStream_t st);
cudaError_t launch_scatter(const Params& p, int num_sms, cudaStream_t st);
cudaError_t launch_rank(const Params& p, int num_sms, cudaStream_t st);
cudaError_t launch_finalize(const Params& p, int num_sms, cudaStream_t st);
cudaError_t launch_zero(void* ptr, size_t bytes, cudaStream_t st);

}  // namespace mmbev
