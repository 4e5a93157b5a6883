// Stages 2-7: voxel cap and canonical order (S4 of the path).
//
// The voxels of a frame must come out in ascending linear index, and when a
// frame has more than max_voxels voxels only the max_voxels smallest by
// (minimum ROI rank, lin) survive (Sec. IV-F hard voxelization; Sec. IV-C
// mandatory ROIs first). No comparison sort is used. Linear indices are cut
// into buckets of 2^LB consecutive cells; the rank of a voxel among the
// frame's voxels is
//     (voxels in earlier buckets of the frame) + (set bits below it in its
//      bucket's occupancy bitmap),
// the first term from one exclusive scan over all buckets, the second from a
// popcount over a per-warp shared-memory bitmap.
//
// Capped frames: a histogram of minimum ranks gives the threshold rank r*
// (the smallest rank whose cumulative count reaches max_voxels) and the
// quota q of rank-r* voxels that still fit. Voxels below r* are all kept,
// those above are dropped, and of the rank-r* ("tie") voxels the q smallest
// by lin are kept. Each bucket counter carries two 32-bit counts (below in
// the low half, tie in the high half), scanned together as one u64, so a
// voxel's output position is A + min(c, q) where A counts below-voxels and c
// counts tie-voxels with a smaller lin in the same frame.
//
//   census          (stage 2)  per voxel: bucket counts of uncapped frames,
//                              rank histogram of capped frames
//   frames          (stage 3)  per frame: r*, q, kept count, output base
//   capped census   (stage 4)  per voxel of a capped frame: class and bucket count
//   scan            (stage 5)  decoupled look-back exclusive scan of the counters
//   scatter         (stage 6)  voxel ids grouped by bucket
//   rank            (stage 7)  per bucket: bitmaps, popcounts, output position,
//                              coordinates
#include "mmbev_internal.cuh"

namespace mmbev {
namespace {

constexpr int kThreads = 256;
constexpr int kRankWarps = 8;
constexpr int kBmWords = (1 << kBucketLog2Max) / 32;

__device__ __forceinline__ void zero_slot(const Params& p, uint32_t h) {
    uint4* s = reinterpret_cast<uint4*>(p.table + (size_t)h * p.slot_stride);
    const uint32_t n = p.slot_stride / 16;
    for (uint32_t i = 0; i < n; ++i) s[i] = make_uint4(0u, 0u, 0u, 0u);
}

__device__ __forceinline__ uint32_t slot_minrank(const Params& p, uint32_t h) {
    return 0xFFFFFFFFu - ld_cg(slot_rank(p, h));
}

// Warp-aggregated atomicAdd of `add` on bcnt[b] for the active lanes in
// `am`; returns this lane's position in the bucket (old lo + old hi + the
// group lanes before it).
__device__ __forceinline__ uint32_t bucket_add(const Params& p, uint32_t am, uint32_t b,
                                               unsigned long long add, int lane) {
    const uint32_t grp = __match_any_sync(am, b);
    const int leader = __ffs(grp) - 1;
    // sum of the group's adds: lanes add either 1 or 1<<32
    const uint32_t lo_n = __popc(__ballot_sync(grp, add == 1ull) & grp);
    const uint32_t hi_n = __popc(grp) - lo_n;
    unsigned long long old = 0ull;
    if (lane == leader)
        old = atomicAdd(&p.bcnt[b], (unsigned long long)lo_n + ((unsigned long long)hi_n << 32));
    old = __shfl_sync(grp, old, leader);
    const uint32_t base = (uint32_t)old + (uint32_t)(old >> 32);
    return base + __popc(grp & ((1u << lane) - 1u));
}

// ---------------------------------------------------------------- stage 2
__global__ void __launch_bounds__(kThreads) k_census(Params p) {
    const uint32_t U = ld_cg(&p.hdr->num_occ);
    const int lane = threadIdx.x & 31;
    const uint32_t gw = (blockIdx.x * blockDim.x + threadIdx.x) >> 5;
    const uint32_t nw = (gridDim.x * blockDim.x) >> 5;
    for (uint32_t base = gw * 32u; base < U; base += nw * 32u) {
        const uint32_t d = base + lane;
        const bool act = d < U;
        uint32_t b = 0, f = 0, h = 0;
        bool capped = false;
        if (act) {
            h = p.occ[d];
            const unsigned long long key = ld_cg(slot_key(p, h)) - 1ull;
            f = (uint32_t)(key >> 32);
            const uint32_t lin = (uint32_t)key;
            b = f * p.buckets_per_frame + (lin >> p.bucket_log2);
            capped = ld_cg(&p.frame_u[f]) > (uint32_t)p.max_voxels;
            p.d_bucket[d] = b;
        }
        const uint32_t am = __ballot_sync(0xFFFFFFFFu, act && !capped);
        if (act && !capped) {
            p.d_pos[d] = bucket_add(p, am, b, 1ull, lane);
        } else if (act) {
            p.d_pos[d] = kUnset;
            const uint32_t r = slot_minrank(p, h);
            atomicAdd(&p.hist[p.frame_roi_off[f] + r], 1u);
        }
    }
}

// ---------------------------------------------------------------- stage 3
__global__ void __launch_bounds__(1024) k_frames(Params p) {
    __shared__ uint32_t s_nvox[kMaxFrames];
    __shared__ uint32_t s_wsum[32];
    const int t = threadIdx.x, lane = t & 31, warp = t >> 5;
    const uint32_t maxv = (uint32_t)p.max_voxels;
    uint32_t any_capped = 0;
    for (int f = warp; f < p.num_frames; f += 32) {
        const uint32_t u = p.frame_u[f];
        FrameInfo fi{};
        if (u <= maxv) {
            fi.capped = 0;
            fi.rstar = 0xFFFFFFFFu;
            fi.q = 0;
            fi.nvox = u;
        } else {
            fi.capped = 1;
            fi.nvox = maxv;
            const int r0 = p.frame_roi_off[f];
            const int rn = p.frame_roi_off[f + 1] - r0;
            uint32_t run = 0;  // voxels with rank below this chunk
            fi.rstar = (uint32_t)rn;
            fi.q = 0;
            for (int c = 0; c < rn; c += 32) {
                const uint32_t v = (c + lane < rn) ? p.hist[r0 + c + lane] : 0u;
                uint32_t inc = v;
#pragma unroll
                for (int o = 1; o < 32; o <<= 1) {
                    const uint32_t x = __shfl_up_sync(0xFFFFFFFFu, inc, o);
                    if (lane >= o) inc += x;
                }
                // first lane whose cumulative count reaches maxv
                const uint32_t hit = __ballot_sync(0xFFFFFFFFu, c + lane < rn && run + inc >= maxv);
                if (hit) {
                    const int l = __ffs(hit) - 1;
                    const uint32_t excl = __shfl_sync(0xFFFFFFFFu, inc - v, l);
                    fi.rstar = (uint32_t)(c + l);
                    fi.q = maxv - (run + excl);
                    break;
                }
                run += __shfl_sync(0xFFFFFFFFu, inc, 31);
            }
            any_capped = 1;
        }
        if (lane == 0) {
            s_nvox[f] = fi.nvox;
            p.finfo[f] = fi;
        }
    }
    if (lane == 0 && any_capped) atomicOr(&p.hdr->any_capped, 1u);
    __syncthreads();
    // exclusive scan of s_nvox over frames (one chunk of 1024 at a time)
    uint32_t carry = 0;
    for (int c = 0; c < p.num_frames; c += 1024) {
        const int f = c + t;
        const uint32_t v = f < p.num_frames ? s_nvox[f] : 0u;
        uint32_t inc = v;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const uint32_t x = __shfl_up_sync(0xFFFFFFFFu, inc, o);
            if (lane >= o) inc += x;
        }
        if (lane == 31) s_wsum[warp] = inc;
        __syncthreads();
        if (warp == 0) {
            uint32_t w = s_wsum[lane];
#pragma unroll
            for (int o = 1; o < 32; o <<= 1) {
                const uint32_t x = __shfl_up_sync(0xFFFFFFFFu, w, o);
                if (lane >= o) w += x;
            }
            s_wsum[lane] = w;  // inclusive warp totals
        }
        __syncthreads();
        const uint32_t wexcl = warp > 0 ? s_wsum[warp - 1] : 0u;
        if (f < p.num_frames) {
            const uint32_t vb = carry + wexcl + inc - v;
            p.finfo[f].vbase = vb;
            p.out_nvox[f] = (int32_t)v;
        }
        carry += s_wsum[31];
        __syncthreads();
    }
    if (t == 0) p.hdr->total_kept = carry;
}

// ---------------------------------------------------------------- stage 4
__global__ void __launch_bounds__(kThreads) k_capped_census(Params p) {
    if (ld_cg(&p.hdr->any_capped) == 0u) return;
    const uint32_t U = ld_cg(&p.hdr->num_occ);
    const int lane = threadIdx.x & 31;
    const uint32_t gw = (blockIdx.x * blockDim.x + threadIdx.x) >> 5;
    const uint32_t nw = (gridDim.x * blockDim.x) >> 5;
    for (uint32_t base = gw * 32u; base < U; base += nw * 32u) {
        const uint32_t d = base + lane;
        bool mine = false;
        uint32_t b = 0;
        unsigned long long add = 0ull;
        if (d < U) {
            b = p.d_bucket[d];
            const uint32_t f = b / p.buckets_per_frame;
            const FrameInfo fi = p.finfo[f];
            if (fi.capped) {
                const uint32_t h = p.occ[d];
                const uint32_t r = slot_minrank(p, h);
                if (r < fi.rstar) { mine = true; add = 1ull; }
                else if (r == fi.rstar) { mine = true; add = 1ull << 32; }
                else { p.d_pos[d] = kUnset; zero_slot(p, h); }  // dropped: release the slot
            }
        }
        const uint32_t am = __ballot_sync(0xFFFFFFFFu, mine);
        if (mine) p.d_pos[d] = bucket_add(p, am, b, add, lane);
    }
}

// ---------------------------------------------------------------- stage 5
__device__ __forceinline__ void st_release(uint32_t* a, uint32_t v) {
    asm volatile("st.release.gpu.global.u32 [%0], %1;" ::"l"(a), "r"(v) : "memory");
}
__device__ __forceinline__ uint32_t ld_acquire(const uint32_t* a) {
    uint32_t v;
    asm volatile("ld.acquire.gpu.global.u32 %0, [%1];" : "=r"(v) : "l"(a) : "memory");
    return v;
}

__global__ void __launch_bounds__(kScanThreads) k_scan(Params p) {
    __shared__ unsigned long long s_wsum[kScanThreads / 32];
    __shared__ unsigned long long s_prefix;
    __shared__ uint32_t s_tile;
    const int t = threadIdx.x, lane = t & 31, warp = t >> 5;
    if (t == 0) s_tile = atomicAdd(&p.hdr->scan_ticket, 1u);
    __syncthreads();
    const uint32_t tile = s_tile;
    const uint64_t L = (uint64_t)p.num_buckets + 1;  // exclusive scan incl. the total slot
    const uint64_t i0 = (uint64_t)tile * kScanTile + (uint64_t)t * kScanPerThread;
    unsigned long long v[kScanPerThread];
    unsigned long long tsum = 0ull;
#pragma unroll
    for (int k = 0; k < kScanPerThread; ++k) {
        v[k] = (i0 + k < L) ? p.bcnt[i0 + k] : 0ull;
        tsum += v[k];
    }
    unsigned long long inc = tsum;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        const unsigned long long x = __shfl_up_sync(0xFFFFFFFFu, inc, o);
        if (lane >= o) inc += x;
    }
    if (lane == 31) s_wsum[warp] = inc;
    __syncthreads();
    unsigned long long wexcl = 0ull, total = 0ull;
#pragma unroll
    for (int w = 0; w < kScanThreads / 32; ++w) {
        if (w < warp) wexcl += s_wsum[w];
        total += s_wsum[w];
    }
    if (t == 0) {
        unsigned long long prefix = 0ull;
        if (tile == 0) {
            p.scan_inc[0] = total;
            st_release(&p.scan_flag[0], 2u);
        } else {
            p.scan_agg[tile] = total;
            st_release(&p.scan_flag[tile], 1u);
            int64_t j = (int64_t)tile - 1;
            uint32_t spins = 0;
            while (j >= 0) {
                const uint32_t fl = ld_acquire(&p.scan_flag[j]);
                if (fl == 2u) { prefix += ld_cg(&p.scan_inc[j]); break; }
                if (fl == 1u) { prefix += ld_cg(&p.scan_agg[j]); --j; continue; }
                if (++spins > kSpinLimit) { set_status(p.hdr, MMBEV_DEV_WAIT_TIMEOUT); break; }
                __nanosleep(32);
            }
            p.scan_inc[tile] = prefix + total;
            st_release(&p.scan_flag[tile], 2u);
        }
        s_prefix = prefix;
    }
    __syncthreads();
    unsigned long long run = s_prefix + wexcl + inc - tsum;
#pragma unroll
    for (int k = 0; k < kScanPerThread; ++k) {
        if (i0 + k < L) p.bcnt[i0 + k] = run;
        run += v[k];
    }
}

// ---------------------------------------------------------------- stage 6
__global__ void __launch_bounds__(kThreads) k_scatter(Params p) {
    const uint32_t U = ld_cg(&p.hdr->num_occ);
    const uint32_t gs = gridDim.x * blockDim.x;
    for (uint32_t d = blockIdx.x * blockDim.x + threadIdx.x; d < U; d += gs) {
        const uint32_t pos = p.d_pos[d];
        if (pos == kUnset) continue;
        const unsigned long long o = p.bcnt[p.d_bucket[d]];
        const uint64_t at = (uint64_t)(uint32_t)o + (uint64_t)(uint32_t)(o >> 32) + pos;
        if (at < U) p.items[at] = d;
        else set_status(p.hdr, MMBEV_DEV_BOUNDS);
    }
}

// ---------------------------------------------------------------- stage 7
__global__ void __launch_bounds__(kRankWarps * 32) k_rank(Params p) {
    __shared__ uint32_t s_below[kRankWarps][kBmWords];
    __shared__ uint32_t s_tie[kRankWarps][kBmWords];
    __shared__ uint16_t s_pb[kRankWarps][kBmWords];
    __shared__ uint16_t s_pt[kRankWarps][kBmWords];
    const int lane = threadIdx.x & 31, wl = threadIdx.x >> 5;
    uint32_t* bm_below = s_below[wl];
    uint32_t* bm_tie = s_tie[wl];
    uint16_t* pb = s_pb[wl];
    uint16_t* pt = s_pt[wl];
    const int nwords = 1 << (p.bucket_log2 - 5);
    const int wpl = (nwords + 31) / 32;  // words per lane
    const uint32_t lbmask = (1u << p.bucket_log2) - 1u;
    const uint32_t U = ld_cg(&p.hdr->num_occ);
    const uint32_t nx = p.dims[0], ny = p.dims[1];
    const uint32_t gw = blockIdx.x * kRankWarps + wl;
    const uint32_t nw = gridDim.x * kRankWarps;
    for (uint32_t b = gw; b < p.num_buckets; b += nw) {
        const unsigned long long o0 = p.bcnt[b], o1 = p.bcnt[b + 1];
        const uint32_t start = (uint32_t)o0 + (uint32_t)(o0 >> 32);
        const uint32_t end = (uint32_t)o1 + (uint32_t)(o1 >> 32);
        if (end <= start) continue;
        if (end > U) { if (lane == 0) set_status(p.hdr, MMBEV_DEV_BOUNDS); continue; }
        const uint32_t f = b / p.buckets_per_frame;
        const FrameInfo fi = p.finfo[f];
        const unsigned long long fb = p.bcnt[(size_t)f * p.buckets_per_frame];
        const uint32_t a0 = (uint32_t)o0 - (uint32_t)fb;
        const uint32_t c0 = (uint32_t)(o0 >> 32) - (uint32_t)(fb >> 32);
        for (int w = lane; w < nwords; w += 32) { bm_below[w] = 0u; bm_tie[w] = 0u; }
        __syncwarp();
        for (uint32_t i = start + lane; i < end; i += 32) {
            const uint32_t d = p.items[i];
            if (d >= U) { set_status(p.hdr, MMBEV_DEV_BOUNDS); continue; }
            const uint32_t h = p.occ[d];
            const uint32_t lin = (uint32_t)(ld_cg(slot_key(p, h)) - 1ull);
            const uint32_t bit = lin & lbmask;
            const bool tie = fi.capped && slot_minrank(p, h) == fi.rstar;
            atomicOr(tie ? &bm_tie[bit >> 5] : &bm_below[bit >> 5], 1u << (bit & 31));
        }
        __syncwarp();
        // per-word exclusive prefix popcounts
        uint32_t sb = 0, st = 0;
        for (int k = 0; k < wpl; ++k) {
            const int w = lane * wpl + k;
            if (w < nwords) { sb += __popc(bm_below[w]); st += __popc(bm_tie[w]); }
        }
        uint32_t ib = sb, it = st;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const uint32_t xb = __shfl_up_sync(0xFFFFFFFFu, ib, o);
            const uint32_t xt = __shfl_up_sync(0xFFFFFFFFu, it, o);
            if (lane >= o) { ib += xb; it += xt; }
        }
        uint32_t rb = ib - sb, rt = it - st;
        for (int k = 0; k < wpl; ++k) {
            const int w = lane * wpl + k;
            if (w < nwords) {
                pb[w] = (uint16_t)rb;
                pt[w] = (uint16_t)rt;
                rb += __popc(bm_below[w]);
                rt += __popc(bm_tie[w]);
            }
        }
        __syncwarp();
        for (uint32_t i = start + lane; i < end; i += 32) {
            const uint32_t d = p.items[i];
            if (d >= U) continue;
            const uint32_t h = p.occ[d];
            const uint32_t lin = (uint32_t)(ld_cg(slot_key(p, h)) - 1ull);
            const uint32_t bit = lin & lbmask;
            const uint32_t w = bit >> 5, m = (1u << (bit & 31)) - 1u;
            const bool tie = fi.capped && slot_minrank(p, h) == fi.rstar;
            const uint32_t A = a0 + pb[w] + __popc(bm_below[w] & m);
            const uint32_t c = c0 + pt[w] + __popc(bm_tie[w] & m);
            bool kept;
            uint32_t vid;
            if (tie) { kept = c < fi.q; vid = A + c; }
            else { kept = true; vid = A + (c < fi.q ? c : fi.q); }
            if (kept && vid < fi.nvox) {
                p.vid_slot[fi.vbase + vid] = h;
                const size_t row = (size_t)f * (uint32_t)p.max_voxels + vid;
                const uint32_t cx = lin % nx;
                const uint32_t cy = (lin / nx) % ny;
                const uint32_t cz = lin / (nx * ny);
                p.out_coords[row * 3 + 0] = (int32_t)cz;
                p.out_coords[row * 3 + 1] = (int32_t)cy;
                p.out_coords[row * 3 + 2] = (int32_t)cx;
            } else {
                if (kept) set_status(p.hdr, MMBEV_DEV_BOUNDS);
                zero_slot(p, h);  // dropped by the cap: release the slot
            }
        }
        __syncwarp();
    }
}

}  // namespace

cudaError_t launch_census(const Params& p, int num_sms, cudaStream_t st) {
    k_census<<<num_sms * 4, kThreads, 0, st>>>(p);
    return cudaGetLastError();
}

cudaError_t launch_frames(const Params& p, cudaStream_t st) {
    k_frames<<<1, 1024, 0, st>>>(p);
    return cudaGetLastError();
}

cudaError_t launch_capped_census(const Params& p, int num_sms, cudaStream_t st) {
    k_capped_census<<<num_sms * 4, kThreads, 0, st>>>(p);
    return cudaGetLastError();
}

cudaError_t launch_scan(const Params& p, cudaStream_t st) {
    k_scan<<<p.scan_tiles, kScanThreads, 0, st>>>(p);
    return cudaGetLastError();
}

cudaError_t launch_scatter(const Params& p, int num_sms, cudaStream_t st) {
    k_scatter<<<num_sms * 4, kThreads, 0, st>>>(p);
    return cudaGetLastError();
}

cudaError_t launch_rank(const Params& p, int num_sms, cudaStream_t st) {
    uint32_t blocks = (p.num_buckets + kRankWarps - 1) / kRankWarps;
    const uint32_t cap = (uint32_t)num_sms * 8u;
    if (blocks > cap) blocks = cap;
    if (blocks == 0) blocks = 1;
    k_rank<<<blocks, kRankWarps * 32, 0, st>>>(p);
    return cudaGetLastError();
}

}  // namespace mmbev
