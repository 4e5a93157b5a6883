// Stage 0: per-call preparation.
//
// One block per frame derives the prepared ROI table (cos/sin of yaw in
// double, rounded to fp32; half-extents grown by the margin, Eq. 1) and the
// frame's coarse BEV candidate mask: for every coarse cell, a bit per ROI
// whose margin-grown box may touch the cell. The mask is conservative (the
// exact per-point test of Alg. 1 follows), so it only prunes work. The other
// blocks copy the host offsets into the workspace and zero the per-call
// counters and the digit histograms.
#include <atomic>
#include <cmath>

#include "mmbev_internal.cuh"

namespace mmbev {
namespace {

constexpr int kPrepThreads = 512;
constexpr int kZeroBlocks = 64;

// Inclusive cell range of one ROI's padded bounding box, or an empty range.
// Computed in fp32: the 5 cm pad (plus a relative term) dwarfs the rounding
// of this bound, of the exact test and of the cell index a point computes.
struct CellRange { int16_t i0, i1, j0, j1; };

__device__ CellRange roi_cells(const Params& p, const RoiPrep& r) {
    CellRange cr{1, 0, 1, 0};
    // NaN anywhere makes the exact test false for every point: no cells.
    if (isnan(r.c) || isnan(r.s) || isnan(r.hl) || isnan(r.hw) || isnan(r.cx) || isnan(r.cy))
        return cr;
    const float ex = fabsf(r.c) * r.hl + fabsf(r.s) * r.hw;
    const float ey = fabsf(r.s) * r.hl + fabsf(r.c) * r.hw;
    const int G = p.coarse;
    float x0 = r.cx - ex, x1 = r.cx + ex, y0 = r.cy - ey, y1 = r.cy + ey;
    if (!(isfinite(x0) && isfinite(x1) && isfinite(y0) && isfinite(y1))) {
        // infinite extents or centre: mark the whole grid (conservative)
        cr.i0 = 0; cr.i1 = (int16_t)(G - 1); cr.j0 = 0; cr.j1 = (int16_t)(G - 1);
        return cr;
    }
    const float span = fabsf(p.rmin[0]) + fabsf(p.rmax[0]) + fabsf(p.rmin[1]) + fabsf(p.rmax[1]);
    const float pad = 0.05f + 1e-4f * (fabsf(r.cx) + fabsf(r.cy) + fabsf(ex) + fabsf(ey) + span);
    x0 -= pad; x1 += pad; y0 -= pad; y1 += pad;
    if (x1 < x0 || y1 < y0) return cr;
    const float fi0 = floorf((x0 - p.rmin[0]) * p.coarse_inv[0]);
    const float fi1 = floorf((x1 - p.rmin[0]) * p.coarse_inv[0]);
    const float fj0 = floorf((y0 - p.rmin[1]) * p.coarse_inv[1]);
    const float fj1 = floorf((y1 - p.rmin[1]) * p.coarse_inv[1]);
    if (fi1 < 0.f || fj1 < 0.f || fi0 > (float)(G - 1) || fj0 > (float)(G - 1)) return cr;
    cr.i0 = (int16_t)fmaxf(fi0, 0.f); cr.i1 = (int16_t)fminf(fi1, (float)(G - 1));
    cr.j0 = (int16_t)fmaxf(fj0, 0.f); cr.j1 = (int16_t)fminf(fj1, (float)(G - 1));
    return cr;
}

__global__ void __launch_bounds__(kPrepThreads)
k_prep(Params p, const __grid_constant__ HostDesc d) {
    extern __shared__ uint32_t s_mask[];  // [coarse^2 * mask_words] for frame blocks
    __shared__ CellRange s_rng[kMaxRoisPerFrame];
    const int t = threadIdx.x;
    if ((int)blockIdx.x < p.num_frames) {
        const int f = blockIdx.x;
        const int r0 = d.frame_roi_off[f];
        const int rn = d.frame_roi_off[f + 1] - r0;
        const int g2 = p.coarse * p.coarse;
        const int W = p.mask_words;
        for (int i = t; i < g2 * W; i += blockDim.x) s_mask[i] = 0u;
        // one thread per ROI: cos/sin of the yaw in double, rounded to fp32
        // (the definition), half-extents grown by the margin, cell range
        for (int r = t; r < rn; r += blockDim.x) {
            const RoiPrep rp = prep_roi(p.rois[r0 + r], p.margin);
            p.roi_prep[r0 + r] = rp;
            s_rng[r] = roi_cells(p, rp);
        }
        __syncthreads();
        // one warp per ROI sets its bit in every cell of its range
        const int warp = t >> 5, lane = t & 31, nwarps = blockDim.x >> 5;
        for (int r = warp; r < rn; r += nwarps) {
            const CellRange cr = s_rng[r];
            const int ni = cr.i1 - cr.i0 + 1, nj = cr.j1 - cr.j0 + 1;
            if (ni <= 0 || nj <= 0) continue;
            const uint32_t bit = 1u << (r & 31);
            const int w = r >> 5;
            for (int k = lane; k < ni * nj; k += 32) {
                const int i = cr.i0 + k % ni, j = cr.j0 + k / ni;
                atomicOr(&s_mask[(j * p.coarse + i) * W + w], bit);
            }
        }
        __syncthreads();
        uint4* gm = reinterpret_cast<uint4*>(p.masks + (size_t)f * g2 * W);
        const uint4* sm4 = reinterpret_cast<const uint4*>(s_mask);
        for (int i = t; i < g2 * W / 4; i += blockDim.x) gm[i] = sm4[i];
        return;
    }
    // Housekeeping blocks: grid-stride over the zero/copy work.
    const int zb = blockIdx.x - p.num_frames;
    const int nz = gridDim.x - p.num_frames;
    const size_t gt = (size_t)zb * blockDim.x + t;
    const size_t gs = (size_t)nz * blockDim.x;
    if (gt < sizeof(Header) / 4 && !(gt == 0 && p.keep_status))   // word 0: the status
        reinterpret_cast<uint32_t*>(p.hdr)[gt] = gt == 0 ? p.inject_status : 0u;
    if (gt == 0 && p.keep_status && p.inject_status) set_status(p.hdr, p.inject_status);
    for (size_t i = gt; i <= (size_t)p.num_sweeps; i += gs) p.sweep_off[i] = d.sweep_off[i];
    for (size_t i = gt; i <= (size_t)p.num_frames; i += gs) {
        p.frame_sweep_off[i] = d.frame_sweep_off[i];
        p.frame_roi_off[i] = d.frame_roi_off[i];
    }
    for (size_t s = gt; s < (size_t)p.num_sweeps; s += gs) {
        // frame of sweep s: last f with frame_sweep_off[f] <= s
        int lo = 0, hi = p.num_frames;  // invariant: fso[lo] <= s < fso[hi]
        while (hi - lo > 1) {
            const int mid = (lo + hi) >> 1;
            if (d.frame_sweep_off[mid] <= (int)s) lo = mid; else hi = mid;
        }
        p.sweep_frame[s] = lo;
    }
    if (p.cls_cnt)
        for (size_t i = gt; i < (size_t)kMaxClsGrid; i += gs) p.cls_cnt[i] = 0u;
    // the per-frame counts and digit histograms start at zero
    if (p.hist)
        for (size_t i = gt; i < (size_t)p.num_frames * kMaxPasses * kDigits; i += gs) p.hist[i] = 0u;
    if (p.fcnt)
        for (size_t i = gt; i < (size_t)p.num_frames; i += gs) p.fcnt[i] = 0u;
    if (p.ftot)
        for (size_t i = gt; i < (size_t)p.num_frames; i += gs) p.ftot[i] = 0u;
}

// One thread per ROI: the prepared form the classify pass tests against.
__global__ void k_prep_rois(const mmbev_roi_t* rois, int32_t n, float margin, float* out) {
    const int i = blockIdx.x * blockDim.x + threadIdx.x;
    if (i >= n) return;
    const RoiPrep rp = prep_roi(rois[i], margin);
    float* o = out + (size_t)i * 6;
    o[0] = rp.cx; o[1] = rp.cy; o[2] = rp.c; o[3] = rp.s; o[4] = rp.hl; o[5] = rp.hw;
}

__global__ void k_zero(uint4* ptr, size_t n16, uint8_t* tail, size_t ntail) {
    const size_t gs = (size_t)gridDim.x * blockDim.x;
    for (size_t i = (size_t)blockIdx.x * blockDim.x + threadIdx.x; i < n16; i += gs)
        ptr[i] = make_uint4(0u, 0u, 0u, 0u);
    if (blockIdx.x == 0)
        for (size_t i = threadIdx.x; i < ntail; i += blockDim.x) tail[i] = 0;
}

}  // namespace

// Largest coarse mask a frame block holds in shared memory: 8,192 words (the
// coarse grid shrinks as the ROI count grows).
constexpr int kPrepSmemMax = 8192 * 4;

cudaError_t launch_prep(const Params& p, const HostDesc& d, cudaStream_t st) {
    // Raise the dynamic shared memory limit once per device (outside any
    // stream capture that may follow).
    static std::atomic<int> configured[64];
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    if (dev < 0 || dev >= 64 || !configured[dev].load(std::memory_order_acquire)) {
        e = cudaFuncSetAttribute(k_prep, cudaFuncAttributeMaxDynamicSharedMemorySize, kPrepSmemMax);
        if (e != cudaSuccess) return e;
        if (dev >= 0 && dev < 64) configured[dev].store(1, std::memory_order_release);
    }
    const size_t smem = (size_t)p.coarse * p.coarse * p.mask_words * sizeof(uint32_t);
    if (smem > (size_t)kPrepSmemMax) return cudaErrorInvalidValue;
    k_prep<<<p.num_frames + kZeroBlocks, kPrepThreads, smem, st>>>(p, d);
    return cudaGetLastError();
}

cudaError_t launch_prep_rois(const mmbev_roi_t* rois, int32_t n, float margin, float* out,
                             cudaStream_t st) {
    if (n <= 0) return cudaSuccess;
    k_prep_rois<<<(unsigned)((n + 255) / 256), 256, 0, st>>>(rois, n, margin, out);
    return cudaGetLastError();
}

cudaError_t launch_zero(void* ptr, size_t bytes, cudaStream_t st) {
    if (bytes == 0) return cudaSuccess;
    const size_t n16 = bytes / 16;
    uint8_t* tail = static_cast<uint8_t*>(ptr) + n16 * 16;
    const size_t blocks = n16 / 256 + 1 < 4096 ? n16 / 256 + 1 : 4096;
    k_zero<<<(unsigned)blocks, 256, 0, st>>>(static_cast<uint4*>(ptr), n16, tail, bytes - n16 * 16);
    return cudaGetLastError();
}

}  // namespace mmbev
