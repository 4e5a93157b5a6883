// Internal declarations shared by the kernels of libmmbev (sm_103a).
//
// Data layout (one call):
//   points      caller's float32 [N][5] AoS, streamed once by the classify
//               kernel through a ring of (up to four) 40 KB shared-memory
//               tiles, each tile moved by eight 5 KB cp.async.bulk (TMA)
//               copies.
//   records     workspace, 32 B per kept point, at position region*32 + (its
//               rank among the kept points of its 32-point region):
//               {x', y', z', intensity} {dt, ROI rank, -, -}. Region g holds
//               points 32g .. 32g+31, so positions increase with the point
//               index and "first K by position" is "first K by index".
//   rcnt, ckey  workspace, per region its kept points (one byte), and per
//               record position the kept point's frame and lin
//               (frame << 32 | lin), both written by classify.
//   keys/vals   workspace, two buffers of M lins and M record positions: the
//               kept points in position order (the compaction stage), so
//               frame by frame, then after each 9-bit LSD radix pass, done
//               within each frame, sorted by one more digit. Every pass is
//               stable, so the last leaves each voxel's points together, in
//               ascending lin, in ascending position. Frame f's items start
//               at the sum of the kept counts fcnt of the frames before it.
//   vdesc       workspace, voxel v of frame f at (frame f's first item) + v,
//               voxels in ascending lin: {first item, end item, lin,
//               minimum ROI rank}, the items being the voxel's run.
//   ftot        workspace [F], voxels of each frame.
//   workspace   Header + per-call arrays (see Layout in api.cu).
#pragma once

#include <cstdint>
#include <cuda_runtime.h>

#include "mmbev.h"

namespace mmbev {

constexpr int kMaxSweeps = MMBEV_MAX_SWEEPS;
constexpr int kMaxFrames = MMBEV_MAX_FRAMES;
constexpr int kMaxRoisPerFrame = MMBEV_MAX_ROIS_PER_FRAME;
constexpr int kMaxK = MMBEV_MAX_PTS_PER_VOXEL;

// Point tiles: 2048 points (40 KB) per tile, 64 regions of 32 points.
constexpr int kTile = 2048;
constexpr int kTileBytes = kTile * 5 * 4;
constexpr int kRegion = 32;
// Points of one call: whole tiles of record slots stay below 2^32.
constexpr int64_t kMaxPoints = MMBEV_MAX_POINTS;
static_assert(kMaxPoints % kTile == 0 && kMaxPoints + kTile == (int64_t{1} << 32), "point limit");

// Classify blocks (one per SM, at most this many).
constexpr int kMaxClsGrid = 1000;

// The kept points are sorted by lin within each frame with 9-bit digits:
// at most four passes for grids of up to 2^32 cells.
constexpr int kDigitBits = 9;
constexpr int kDigits = 1 << kDigitBits;
constexpr int kMaxPasses = 4;
constexpr uint32_t kNoLin = 0xFFFFFFFFu;   // above every lin (cells < 2^32)

// Tiles of the radix passes and of the voxel numbering (within one frame).
constexpr uint32_t kSortTile = 4096;
constexpr uint32_t kRunTile = 2048;

// Bounded waits.
constexpr uint32_t kSpinLimit = 1u << 22;

constexpr uint32_t kUnset = 0xFFFFFFFFu;

// Unsigned 32-bit division by a divisor fixed for the whole call, by one
// multiply-high and two shifts (Granlund and Montgomery, "Division by
// Invariant Integers using Multiplication", PLDI 1994, Fig. 4.1): with
// l = ceil(log2 d) and m = floor(2^32 (2^l - d) / d) + 1 (32 bits),
// n / d = (t + ((n - t) >> min(l, 1))) >> max(l - 1, 0), t = mulhi(m, n),
// exact for every 1 <= d < 2^32 and 0 <= n < 2^32.
struct UDiv {
    uint32_t m, s1, s2;
};
inline UDiv udiv_make(uint32_t d) {
    uint32_t l = 0;
    while (l < 32 && (1ull << l) < (uint64_t)d) ++l;
    UDiv u;
    u.m = (uint32_t)((((1ull << l) - d) << 32) / d + 1ull);
    u.s1 = l < 1 ? l : 1u;
    u.s2 = l > 1 ? l - 1u : 0u;
    return u;
}
__device__ __forceinline__ uint32_t udiv(const UDiv& u, uint32_t n) {
    const uint32_t t = __umulhi(u.m, n);
    return (t + ((n - t) >> u.s1)) >> u.s2;
}

// Prepared ROI: centre, cos/sin of yaw, half-extents grown by the margin.
struct __align__(16) RoiPrep {
    float cx, cy, c, s;
    float hl, hw, pad0, pad1;
};

// Workspace header; zeroed by the prep kernel at the start of every call.
struct __align__(16) Header {
    uint32_t status;        // MMBEV_DEV_* bits (first word: read by mmbev_get_status)
    uint32_t num_rec;       // kept points (records) of the call
    uint32_t run_ticket;    // voxel numbering tiles started, in order
    uint32_t sort_ticket[kMaxPasses];   // radix pass tiles started, in order
    uint32_t pad[3];
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
    UDiv div_nx, div_ny;    // division by nx and by ny (voxel coordinates from lin)
    int32_t K;
    int32_t max_voxels;
    uint32_t rho_thr;       // keep a point inside no ROI when its draw's top 24 bits < rho_thr
    uint64_t seed;          // SplitMix64 seed of those draws
    int32_t keep_status = 0;  // prep leaves the status word as it is (later chunks of a call)
    uint32_t inject_status = 0;  // test hook: status bits prep sets as a failure would
    // the sort of the kept points
    int32_t sort_passes;       // 9-bit digits of the largest lin
    // workspace arrays
    Header* hdr;
    int64_t* sweep_off;     // [S+1]
    int32_t* sweep_frame;   // [S]
    int32_t* frame_sweep_off;  // [F+1]
    int32_t* frame_roi_off;    // [F+1]
    RoiPrep* roi_prep;      // [R]
    uint32_t* masks;        // [F][coarse^2][mask_words]
    uint4* records;         // [regions*32][2] kept points' features and rank
    uint32_t* cls_cnt;      // [kMaxClsGrid] kept points of each classify block
    uint32_t* cls_flo;      // [kMaxClsGrid] frame of each classify block's first point
    uint32_t cls_grid;      // classify blocks of the call
    uint32_t num_regions;
    uint32_t rec_cap;       // record positions of the call (regions * 32)
    uint8_t* rcnt;          // [regions] kept points of each region
    unsigned long long* ckey;   // [rec_cap] frame << 32 | lin of the kept point at each position
    uint32_t* key_a;        // [rec_cap] lins, buffer A (the compaction writes it)
    uint32_t* val_a;        // [rec_cap] record positions, buffer A
    uint32_t* key_b;        // [rec_cap] buffer B (with val_b, aliases ckey)
    uint32_t* val_b;
    const uint32_t* skey;   // the sorted buffer (A or B by the pass count)
    const uint32_t* sval;
    uint32_t* fcnt;         // [F] kept points of each frame
    uint32_t* ftot;         // [F] voxels of each frame
    uint32_t* hist;         // [F][kMaxPasses][kDigits] digit histograms of each frame's lins
    unsigned long long* sort_state;   // [2][sort_tiles_cap][kDigits] look-back words of the passes
    unsigned long long* run_state;    // [run_tiles_cap] look-back words of the voxel numbering
    uint32_t sort_tiles_cap;  // tiles of a pass, at most (one more a frame for the ragged ends)
    uint32_t run_tiles_cap;
    uint4* vdesc;           // [rec_cap] per voxel: {first item, end item, lin, minimum rank}
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

// Programmatic dependent launch: wait for the preceding kernel's results.
// No kernel signals its dependents early: they are released as its blocks
// exit, so waiting blocks of the next kernel never take SM slots from blocks
// of the running one, while the next launch is still prepared during the
// running kernel's tail.
__device__ __forceinline__ void pdl_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }

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

// Eq. 1 box of one ROI in the form the inside test takes: cos and sin of the
// yaw evaluated in double and rounded to fp32, half-extents grown by the
// margin (0.5*l + r along the heading, 0.5*w + r across it), in fp32.
__device__ __forceinline__ RoiPrep prep_roi(const mmbev_roi_t& in, float margin) {
    RoiPrep rp;
    rp.cx = in.cx;
    rp.cy = in.cy;
    rp.c = (float)cos((double)in.yaw);
    rp.s = (float)sin((double)in.yaw);
    rp.hl = __fadd_rn(__fmul_rn(0.5f, in.l), margin);
    rp.hw = __fadd_rn(__fmul_rn(0.5f, in.w), margin);
    rp.pad0 = 0.f;
    rp.pad1 = 0.f;
    return rp;
}

// Alg. 1 inside test against one prepared ROI (boundary inclusive).
__device__ __forceinline__ bool roi_contains(const RoiPrep& r, float x, float y) {
    const float dx = __fsub_rn(x, r.cx);
    const float dy = __fsub_rn(y, r.cy);
    const float u = __fadd_rn(__fmul_rn(dx, r.c), __fmul_rn(dy, r.s));
    const float v = __fsub_rn(__fmul_rn(dy, r.c), __fmul_rn(dx, r.s));
    return fabsf(u) <= r.hl && fabsf(v) <= r.hw;
}

// S2, first part: range crop (half-open box) and the point's coarse BEV cell.
// Returns false when the point is out of range; `cell` indexes the frame's
// coarse mask (cells x mask_words words).
__device__ __forceinline__ bool point_cell(const Params& p, float x, float y, float z,
                                           int& cell) {
    if (!((p.rmin[0] <= x) && (x < p.rmax[0]) && (p.rmin[1] <= y) && (y < p.rmax[1]) &&
          (p.rmin[2] <= z) && (z < p.rmax[2])))
        return false;
    const int G = p.coarse;
    int gx = (int)__fmul_rn(__fsub_rn(x, p.rmin[0]), p.coarse_inv[0]);
    int gy = (int)__fmul_rn(__fsub_rn(y, p.rmin[1]), p.coarse_inv[1]);
    gx = min(max(gx, 0), G - 1);
    gy = min(max(gy, 0), G - 1);
    cell = gy * G + gx;
    return true;
}

// Exact ROI test of candidate r (prepared ROIs of the point's frame).
__device__ __forceinline__ bool roi_hit(const RoiPrep* frois, int r, float x, float y) {
    const float4* rp4 = reinterpret_cast<const float4*>(frois + r);
    const float4 a = rp4[0], c = rp4[1];
    RoiPrep rp;
    rp.cx = a.x; rp.cy = a.y; rp.c = a.z; rp.s = a.w; rp.hl = c.x; rp.hw = c.y;
    return roi_contains(rp, x, y);
}

// S2, last part: Eq. 1 voxel index of an in-range point; false when the
// floor lands on or beyond the grid's far face.
__device__ __forceinline__ bool voxel_lin(const Params& p, float x, float y, float z,
                                          uint32_t& lin) {
    const uint32_t cx = __float2uint_rz(__fdiv_rn(__fsub_rn(x, p.rmin[0]), p.vs[0]));
    const uint32_t cy = __float2uint_rz(__fdiv_rn(__fsub_rn(y, p.rmin[1]), p.vs[1]));
    const uint32_t cz = __float2uint_rz(__fdiv_rn(__fsub_rn(z, p.rmin[2]), p.vs[2]));
    if (cx >= p.dims[0] || cy >= p.dims[1] || cz >= p.dims[2]) return false;
    lin = (cz * p.dims[1] + cy) * p.dims[0] + cx;
    return true;
}

// S2 for one compensated point: range crop, coarse-mask candidates, exact
// ROI test in rank order, voxel index. `fmask` is the point's frame's coarse
// mask (coarse^2 cells x mask_words) and `frois` its prepared ROIs. Returns
// true and sets lin, rank when the point is kept.
__device__ __forceinline__ bool classify_point(const Params& p, const uint32_t* fmask,
                                               const RoiPrep* frois, float x, float y, float z,
                                               uint32_t& lin, uint32_t& rank) {
    int cell;
    if (!point_cell(p, x, y, z, cell)) return false;
    const uint32_t* mw = fmask + cell * p.mask_words;
    int hit = -1;
    for (int w = 0; w < p.mask_words && hit < 0; ++w) {
        uint32_t bits = mw[w];
        while (bits) {
            const int b = __ffs(bits) - 1;
            bits &= bits - 1u;
            if (roi_hit(frois, w * 32 + b, x, y)) { hit = w * 32 + b; break; }
        }
    }
    if (hit < 0) return false;
    if (!voxel_lin(p, x, y, z, lin)) return false;
    rank = (uint32_t)hit;
    return true;
}

// Sweep of global point index i: largest s with off[s] <= i (off nondecreasing).
__device__ __forceinline__ int find_sweep(const int64_t* off, int nsweeps, int64_t i) {
    int lo = 0, hi = nsweeps;  // off[lo] <= i < off[hi]
    while (hi - lo > 1) {
        const int mid = (lo + hi) >> 1;
        if (off[mid] <= i) lo = mid; else hi = mid;
    }
    return lo;
}

// The n-th output (n >= 1) of SplitMix64 (Steele, Lea and Flood, OOPSLA
// 2014) started at state `seed`: the finalizer of seed + n * golden gamma.
__device__ __forceinline__ uint64_t splitmix64_nth(uint64_t seed, uint64_t n) {
    uint64_t z = seed + n * 0x9E3779B97F4A7C15ull;
    z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
    z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
    return z ^ (z >> 31);
}

// 64-bit mixer (the SplitMix64 finalizer of Steele, Lea and Flood, 2014).
__device__ __forceinline__ uint64_t mix64(uint64_t z) {
    z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
    z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
    return z ^ (z >> 31);
}

// Home bucket of a hash key in a power-of-two table (mask = buckets - 1).
__device__ __forceinline__ uint32_t slot_home(uint32_t mask, unsigned long long key1) {
    return (uint32_t)mix64(key1) & mask;
}

// Load at L2 (bypassing the non-coherent L1), for words other blocks update.
__device__ __forceinline__ uint32_t ld_cg(const uint32_t* a) { return __ldcg(a); }
__device__ __forceinline__ unsigned long long ld_cg(const unsigned long long* a) {
    return __ldcg(a);
}

// Relaxed load at GPU scope, issued anew every time: for look-back words,
// which carry their flag and value in one word written by one atomic
// exchange, so that nothing else needs ordering after them. Unlike acquire
// loads, several can be in flight at once.
__device__ __forceinline__ unsigned long long ld_relaxed(const unsigned long long* a) {
    unsigned long long v;
    asm volatile("ld.relaxed.gpu.global.u64 %0, [%1];" : "=l"(v) : "l"(a) : "memory");
    return v;
}

// Acquire load at GPU scope, issued anew every time (for polling a word that
// another block publishes).
__device__ __forceinline__ unsigned long long ld_acquire(const unsigned long long* a) {
    unsigned long long v;
    asm volatile("ld.acquire.gpu.global.u64 %0, [%1];" : "=l"(v) : "l"(a) : "memory");
    return v;
}

// ---------------------------------------------------------------- launchers

// All launchers enqueue on `st` and return the launch's error code. `pdl`
// launches the kernel as a programmatic dependent of the preceding one.
cudaError_t launch_prep(const Params& p, const HostDesc& d, cudaStream_t st);
// The prepared form (cx, cy, c, s, hl, hw) of n ROIs into out[n][6].
cudaError_t launch_prep_rois(const mmbev_roi_t* rois, int32_t n, float margin, float* out,
                             cudaStream_t st);
cudaError_t launch_classify(const Params& p, int rmax, int num_sms, bool pdl, cudaStream_t st);
cudaError_t launch_classify_points(const Params& p, cudaStream_t st);
// The stages after classify (csrc/sort.cu): compaction and digit histograms,
// the radix passes, voxel numbering, output rows.
cudaError_t launch_compact(const Params& p, int num_sms, bool pdl, cudaStream_t st);
cudaError_t launch_sort(const Params& p, int num_sms, bool pdl, cudaStream_t st);
cudaError_t launch_runs(const Params& p, int num_sms, bool pdl, cudaStream_t st);
cudaError_t launch_emit(const Params& p, int num_sms, bool pdl, cudaStream_t st);
// Kept rows of frames [f0, f1) of a call's outputs into a packed buffer
// (mmbev_pack_voxels' layout for F frames).
cudaError_t launch_pack(const float* feats, const int32_t* coords, const int32_t* counts,
                        const int32_t* nvox, int32_t F, int32_t f0, int32_t f1,
                        int32_t max_voxels, void* dst, cudaStream_t stream);
int num_sms();   // of the current device, cached
cudaError_t launch_zero(void* ptr, size_t bytes, cudaStream_t st);

// Launch `kern` with an optional programmatic-stream-serialization attribute.
template <typename... KArgs, typename... Args>
cudaError_t launch_k(void (*kern)(KArgs...), dim3 grid, dim3 block, size_t smem,
                     cudaStream_t st, bool pdl, Args&&... args) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = grid;
    cfg.blockDim = block;
    cfg.dynamicSmemBytes = smem;
    cfg.stream = st;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = pdl ? 1 : 0;
    return cudaLaunchKernelEx(&cfg, kern, static_cast<KArgs>(args)...);
}

}  // namespace mmbev
