// Stages 5-9: voxel cap and canonical order (S4 of the path).
//
// The voxels of a frame must come out in ascending linear index, and when a
// frame has more than max_voxels voxels only the max_voxels smallest by
// (minimum ROI rank, lin) survive (Sec. IV-F hard voxelization; Sec. IV-C
// mandatory ROIs first). No comparison sort is used. Linear indices are cut
// into buckets of 2^LB consecutive cells; the rank of a voxel among its
// frame's voxels is
//     (voxels in earlier buckets of the frame) + (set bits below it in its
//      bucket's occupancy bitmap),
// the first term from an exclusive scan of the frame's bucket counters, the
// second from popcounts over a per-warp shared-memory bitmap.
//
// The insert stage already counted every new voxel into its bucket. Frames
// with more voxels than max_voxels ("capped", rare) are recounted with two
// classes: a histogram of minimum ranks gives the threshold rank r* (the
// smallest rank whose cumulative count reaches max_voxels) and the quota q
// of rank-r* voxels that still fit. Voxels below r* are all kept, those
// above are dropped, and of the rank-r* ("tie") voxels the q smallest by lin
// are kept. A capped frame's bucket counters carry two 32-bit counts (below
// in the low half, tie in the high half), scanned together as one u64, so a
// voxel's output position is A + min(c, q), where A counts below-voxels and
// c counts tie-voxels with a smaller lin in the same frame.
//
//   frames          (stage 5)  rank histogram of capped frames, then (the
//                              last block) per frame: r*, q, kept count,
//                              output base, item-segment base
//   capped census   (stage 6)  per voxel of a capped frame: class, bucket count
//   scan            (stage 7)  one block per chunk of 1024 buckets of a frame:
//                              exclusive scan of counters
//   scatter         (stage 8)  voxel ids grouped by bucket
//   rank            (stage 9)  per non-empty bucket: bitmaps, popcounts, output
//                              position, coordinates
#include "mmbev_internal.cuh"

namespace mmbev {
namespace {

constexpr int kThreads = 256;
constexpr int kRankWarps = 8;
constexpr int kBmWords = (1 << kBucketLog2Max) / 32;

// True when some frame has more voxels than max_voxels (every block checks).
__device__ bool block_any_capped(const Params& p) {
    int mine = 0;
    for (int f = threadIdx.x; f < p.num_frames; f += blockDim.x)
        mine |= ld_cg(&p.frame_u[f]) > (uint32_t)p.max_voxels;
    return __syncthreads_or(mine) != 0;
}

// ---------------------------------------------------------------- stage 5
// Per frame: r*, q, kept count, output base, item-segment base, from the
// minimum-rank histogram of the capped frames (F <= 1024 frames). Run by one
// block of any multiple of 32 threads.
__device__ void frames_body(const Params& p, uint32_t* s_nvox, uint32_t* s_u,
                            uint32_t (*s_wsum)[32]) {
    const int t = threadIdx.x, lane = t & 31, warp = t >> 5;
    const int nwarps = (int)(blockDim.x >> 5);
    const uint32_t maxv = (uint32_t)p.max_voxels;
    const int F = p.num_frames;
    uint32_t any_capped = 0;
    for (int f = warp; f < F; f += nwarps) {
        const uint32_t u = ld_cg(&p.frame_u[f]);
        FrameInfo fi{};
        if (u <= maxv) {
            fi.capped = 0;
            fi.rstar = 0xFFFFFFFFu;
            fi.q = 0;
            fi.nvox = u;
        } else {
            fi.capped = 1;
            fi.nvox = maxv;
            // ranks 0 .. R_f (R_f: points kept outside every ROI)
            const int r0 = p.frame_roi_off[f] + f;
            const int rn = p.frame_roi_off[f + 1] - p.frame_roi_off[f] + 1;
            uint32_t run = 0;  // voxels with a rank below this chunk
            fi.rstar = (uint32_t)rn;
            fi.q = 0;
            for (int c = 0; c < rn; c += 32) {
                const uint32_t v = (c + lane < rn) ? ld_cg(&p.hist[r0 + c + lane]) : 0u;
                uint32_t inc = v;
#pragma unroll
                for (int o = 1; o < 32; o <<= 1) {
                    const uint32_t x = __shfl_up_sync(0xFFFFFFFFu, inc, o);
                    if (lane >= o) inc += x;
                }
                // first lane whose cumulative count reaches maxv
                const uint32_t hit =
                    __ballot_sync(0xFFFFFFFFu, c + lane < rn && run + inc >= maxv);
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
            // the capped frame's two-class counters start at zero
            const size_t b0 = (size_t)f * p.buckets_per_frame;
            for (uint32_t b = lane; b < p.buckets_per_frame; b += 32) p.bcnt2[b0 + b] = 0ull;
        }
        if (lane == 0) {
            s_nvox[f] = fi.nvox;
            s_u[f] = u;
            p.finfo[f] = fi;
        }
    }
    if (lane == 0 && any_capped) atomicOr(&p.hdr->any_capped, 1u);
    __syncthreads();
    // exclusive scans over frames of nvox (output rows) and u (item segments)
    uint32_t carry_v = 0, carry_u = 0;
    for (int c = 0; c < F; c += (int)blockDim.x) {
        const int f = c + t;
        const uint32_t v = f < F ? s_nvox[f] : 0u;
        const uint32_t u = f < F ? s_u[f] : 0u;
        uint32_t iv = v, iu = u;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const uint32_t xv = __shfl_up_sync(0xFFFFFFFFu, iv, o);
            const uint32_t xu = __shfl_up_sync(0xFFFFFFFFu, iu, o);
            if (lane >= o) { iv += xv; iu += xu; }
        }
        if (lane == 31) { s_wsum[0][warp] = iv; s_wsum[1][warp] = iu; }
        __syncthreads();
        if (warp == 0) {
            uint32_t a = lane < nwarps ? s_wsum[0][lane] : 0u;
            uint32_t b = lane < nwarps ? s_wsum[1][lane] : 0u;
#pragma unroll
            for (int o = 1; o < 32; o <<= 1) {
                const uint32_t xa = __shfl_up_sync(0xFFFFFFFFu, a, o);
                const uint32_t xb = __shfl_up_sync(0xFFFFFFFFu, b, o);
                if (lane >= o) { a += xa; b += xb; }
            }
            s_wsum[0][lane] = a;
            s_wsum[1][lane] = b;
        }
        __syncthreads();
        if (f < F) {
            const uint32_t wv = warp > 0 ? s_wsum[0][warp - 1] : 0u;
            const uint32_t wu = warp > 0 ? s_wsum[1][warp - 1] : 0u;
            p.finfo[f].vbase = carry_v + wv + iv - v;
            p.finfo[f].ibase = carry_u + wu + iu - u;
            p.out_nvox[f] = (int32_t)v;
        }
        carry_v += s_wsum[0][31];
        carry_u += s_wsum[1][31];
        __syncthreads();
    }
    if (t == 0) p.hdr->total_kept = carry_v;
}

// Every block adds the minimum ranks of its share of the voxels of capped
// frames to their frame's histogram (nothing when no frame is capped); the
// last block to finish, told by a counter, then runs the per-frame stage.
__global__ void __launch_bounds__(kThreads) k_frames(Params p) {
    __shared__ uint32_t s_nvox[kMaxFrames];
    __shared__ uint32_t s_u[kMaxFrames];
    __shared__ uint32_t s_wsum[2][32];
    __shared__ uint32_t s_last;
    pdl_wait();
    if (block_any_capped(p)) {
        const uint32_t U = min(ld_cg(&p.hdr->num_occ), p.occ_cap);
        const uint32_t gs = gridDim.x * blockDim.x;
        for (uint32_t d = blockIdx.x * blockDim.x + threadIdx.x; d < U; d += gs) {
            const uint32_t f = udiv(p.div_bf, p.d_bucket[d]);
            if (ld_cg(&p.frame_u[f]) <= (uint32_t)p.max_voxels) continue;
            const int r0 = p.frame_roi_off[f];
            const uint32_t rn = (uint32_t)(p.frame_roi_off[f + 1] - r0);  // background rank
            const uint32_t r = min(slot_minrank(p, p.occ[d]), rn);
            atomicAdd(&p.hist[r0 + f + r], 1u);
        }
    }
    __threadfence();
    __syncthreads();
    if (threadIdx.x == 0) s_last = atomicAdd(&p.hdr->frames_done, 1u) == gridDim.x - 1u;
    __syncthreads();
    if (!s_last) return;
    __threadfence();
    frames_body(p, s_nvox, s_u, s_wsum);
}

// ---------------------------------------------------------------- stage 6
// Warp-aggregated atomicAdd on cnt[b] for the lanes with `mine` set (1 for a
// rank-below voxel, 1<<32 for a rank-tie voxel); returns each such lane's
// position in the bucket (old lo + old hi + the group lanes before it).
// Called by the whole warp: every collective uses the full mask.
__device__ __forceinline__ uint32_t bucket_add(unsigned long long* cnt, bool mine, uint32_t b,
                                               bool tie, int lane) {
    const uint32_t am = __ballot_sync(0xFFFFFFFFu, mine);
    uint32_t grp = 1u << lane;
    if (mine) grp = __match_any_sync(am, b);
    const int leader = __ffs(grp) - 1;
    const uint32_t ties = __ballot_sync(0xFFFFFFFFu, mine && tie);
    unsigned long long old = 0ull;
    if (mine && lane == leader) {
        const uint32_t hi_n = __popc(grp & ties);
        const uint32_t lo_n = __popc(grp) - hi_n;
        old = atomicAdd(&cnt[b], (unsigned long long)lo_n + ((unsigned long long)hi_n << 32));
    }
    old = __shfl_sync(0xFFFFFFFFu, old, leader);
    const uint32_t base = (uint32_t)old + (uint32_t)(old >> 32);
    return base + __popc(grp & ((1u << lane) - 1u));
}

__global__ void __launch_bounds__(kThreads) k_capped_census(Params p) {
    pdl_wait();
    if (ld_cg(&p.hdr->any_capped) == 0u) return;
    const uint32_t U = min(ld_cg(&p.hdr->num_occ), p.occ_cap);
    const int lane = threadIdx.x & 31;
    const uint32_t gw = (blockIdx.x * blockDim.x + threadIdx.x) >> 5;
    const uint32_t nw = (gridDim.x * blockDim.x) >> 5;
    for (uint32_t base = gw * 32u; base < U; base += nw * 32u) {
        const uint32_t d = base + lane;
        bool mine = false, tie = false;
        uint32_t b = 0;
        if (d < U) {
            b = p.d_bucket[d];
            const FrameInfo fi = p.finfo[udiv(p.div_bf, b)];
            if (fi.capped) {
                const uint32_t h = p.occ[d];
                const uint32_t r = slot_minrank(p, h);
                if (r < fi.rstar) { mine = true; }
                else if (r == fi.rstar) { mine = true; tie = true; }
                else { p.d_pos[d] = kUnset; zero_slot(p, h); }  // dropped: release the slot
            }
        }
        const uint32_t pos = bucket_add(p.bcnt2, mine, b, tie, lane);
        if (mine) p.d_pos[d] = pos;
    }
}

// ---------------------------------------------------------------- stage 7
// boff[b] = sum of the frame's counters before b.
constexpr int kScanThreads = (int)kScanChunk;   // one bucket per thread

// One block per (frame, chunk of kScanChunk buckets): the chunk's base is the
// sum of the frame's earlier chunks (their voxel counts from the compact
// kernel; capped frames sum their two-class counters instead), then a block
// scan gives every bucket its exclusive offset within the frame, and the
// chunk's non-empty buckets are appended to the list with one atomicAdd.
__global__ void __launch_bounds__(kScanThreads) k_scan(Params p) {
    __shared__ unsigned long long s_wsum[kScanThreads / 32];
    __shared__ uint32_t s_nz[kScanThreads / 32];
    __shared__ unsigned long long s_base;
    __shared__ uint32_t s_nzbase;
    pdl_wait();
    const int t = threadIdx.x, lane = t & 31, warp = t >> 5;
    const uint32_t C = p.scan_chunks;
    const uint32_t f = blockIdx.x / C, c = blockIdx.x % C;
    const uint32_t Bf = p.buckets_per_frame;
    const size_t b0 = (size_t)f * Bf;
    const bool capped = p.finfo[f].capped != 0;
    const unsigned long long* src = capped ? p.bcnt2 : p.bcnt;
    // the chunk's base
    unsigned long long part = 0ull;
    if (!capped) {
        for (uint32_t k = t; k < c; k += kScanThreads) part += ld_cg(&p.ctot[f * C + k]);
    } else {
        for (uint32_t k = t; k < c * kScanChunk; k += kScanThreads) part += src[b0 + k];
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) part += __shfl_xor_sync(0xFFFFFFFFu, part, o);
    if (lane == 0) s_wsum[warp] = part;
    __syncthreads();
    if (t == 0) {
        unsigned long long b = 0ull;
        for (int w = 0; w < kScanThreads / 32; ++w) b += s_wsum[w];
        s_base = b;
    }
    __syncthreads();
    const uint32_t i = c * kScanChunk + (uint32_t)t;
    const unsigned long long v = i < Bf ? src[b0 + i] : 0ull;
    const uint32_t nz = v != 0ull;
    unsigned long long inc = v;
    uint32_t nzi = nz;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        const unsigned long long x = __shfl_up_sync(0xFFFFFFFFu, inc, o);
        const uint32_t y = __shfl_up_sync(0xFFFFFFFFu, nzi, o);
        if (lane >= o) { inc += x; nzi += y; }
    }
    if (lane == 31) { s_wsum[warp] = inc; s_nz[warp] = nzi; }
    __syncthreads();
    if (warp == 0) {
        unsigned long long w = s_wsum[lane];
        uint32_t z = s_nz[lane];
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const unsigned long long x = __shfl_up_sync(0xFFFFFFFFu, w, o);
            const uint32_t y = __shfl_up_sync(0xFFFFFFFFu, z, o);
            if (lane >= o) { w += x; z += y; }
        }
        s_wsum[lane] = w;
        s_nz[lane] = z;
        if (lane == 31) s_nzbase = z ? atomicAdd(&p.hdr->num_nonempty, z) : 0u;
    }
    __syncthreads();
    if (i < Bf) {
        p.boff[b0 + i] = s_base + (warp > 0 ? s_wsum[warp - 1] : 0ull) + inc - v;
        if (nz) {
            const uint32_t zpos = s_nzbase + (warp > 0 ? s_nz[warp - 1] : 0u) + nzi - 1u;
            if (zpos < p.num_buckets) p.nonempty[zpos] = (uint32_t)(b0 + i);
        }
    }
}

// ---------------------------------------------------------------- stage 8
__global__ void __launch_bounds__(kThreads) k_scatter(Params p) {
    pdl_wait();
    const uint32_t U = min(ld_cg(&p.hdr->num_occ), p.occ_cap);
    const uint32_t gs = gridDim.x * blockDim.x;
    for (uint32_t d = blockIdx.x * blockDim.x + threadIdx.x; d < U; d += gs) {
        const uint32_t pos = p.d_pos[d];
        if (pos == kUnset) continue;
        const uint32_t b = p.d_bucket[d];
        const unsigned long long o = p.boff[b];
        const uint64_t at = (uint64_t)p.finfo[udiv(p.div_bf, b)].ibase + (uint32_t)o +
                            (uint32_t)(o >> 32) + pos;
        if (at < U) p.items[at] = make_uint2(p.occ[d], p.d_lin[d]);
        else set_status(p.hdr, MMBEV_DEV_BOUNDS);
    }
}

// ---------------------------------------------------------------- stage 9
// Output row `vid` of frame f (call-wide index g) is the voxel in slot h with
// linear index lin: its slot and coordinates.
__device__ __forceinline__ void write_rank(const Params& p, uint32_t g, uint32_t f, uint32_t vid,
                                           uint32_t h, uint32_t lin) {
    p.vid_slot[g] = h;
    // the slot's rank word is not read past this stage: it now holds the
    // voxel's output index, for the finalize stage's heavy role (which starts
    // from the slot)
    *slot_rank(p, h) = g;
    const size_t row = (size_t)f * (uint32_t)p.max_voxels + vid;
    const uint32_t q = udiv(p.div_nx, lin);      // cz * ny + cy
    const uint32_t cz = udiv(p.div_ny, q);
    p.out_coords[row * 3 + 0] = (int32_t)cz;
    p.out_coords[row * 3 + 1] = (int32_t)(q - cz * p.dims[1]);
    p.out_coords[row * 3 + 2] = (int32_t)(lin - q * p.dims[0]);
}

// One warp per non-empty bucket (the scan's list), assigned round-robin.
__global__ void __launch_bounds__(kRankWarps * 32) k_rank(Params p) {
    __shared__ uint32_t s_below[kRankWarps][kBmWords];
    __shared__ uint32_t s_tie[kRankWarps][kBmWords];
    __shared__ uint16_t s_pb[kRankWarps][kBmWords];
    __shared__ uint16_t s_pt[kRankWarps][kBmWords];
    pdl_wait();
    const int lane = threadIdx.x & 31, wl = threadIdx.x >> 5;
    uint32_t* bm_below = s_below[wl];
    uint32_t* bm_tie = s_tie[wl];
    uint16_t* pb = s_pb[wl];
    uint16_t* pt = s_pt[wl];
    const int nwords = 1 << (p.bucket_log2 - 5);
    const int wpl = (nwords + 31) / 32;  // words per lane
    const uint32_t lbmask = (1u << p.bucket_log2) - 1u;
    const uint32_t U = min(ld_cg(&p.hdr->num_occ), p.occ_cap);
    const uint32_t NE = min(ld_cg(&p.hdr->num_nonempty), p.num_buckets);
    const uint32_t gw = blockIdx.x * kRankWarps + wl;
    const uint32_t nw = gridDim.x * kRankWarps;
    for (uint32_t e = gw; e < NE; e += nw) {
        const uint32_t b = p.nonempty[e];
        const uint32_t f = udiv(p.div_bf, b);
        const FrameInfo fi = p.finfo[f];
        const bool capped = fi.capped != 0;
        const unsigned long long cv = capped ? p.bcnt2[b] : p.bcnt[b];
        const uint32_t n = (uint32_t)cv + (uint32_t)(cv >> 32);
        const unsigned long long o = p.boff[b];
        const uint32_t a0 = (uint32_t)o, c0 = (uint32_t)(o >> 32);
        const uint64_t start = (uint64_t)fi.ibase + a0 + c0;
        if (start + n > U) {
            if (lane == 0) set_status(p.hdr, MMBEV_DEV_BOUNDS);
            continue;
        }
        if (!capped && n <= 64) {
            // a bucket of at most 64 voxels in a frame under the cap (95 % of
            // the buckets of 32 nuScenes-shaped frames): lane i holds items i
            // and i + 32, and an item's rank in the bucket is the number of
            // the bucket's (distinct) linear indices below its own, counted
            // over the warp with shuffles
            const uint32_t i1 = (uint32_t)lane + 32u;
            uint2 it0 = make_uint2(0u, 0u), it1 = make_uint2(0u, 0u);
            if ((uint32_t)lane < n) it0 = p.items[start + lane];
            if (i1 < n) it1 = p.items[start + i1];
            const uint32_t k0 = (uint32_t)lane < n ? (it0.y & lbmask) : 0xFFFFFFFFu;
            const uint32_t k1 = i1 < n ? (it1.y & lbmask) : 0xFFFFFFFFu;
            uint32_t r0 = 0, r1 = 0;
            const uint32_t n0 = n < 32u ? n : 32u;
            for (uint32_t j = 0; j < n0; ++j) {
                const uint32_t x = __shfl_sync(0xFFFFFFFFu, k0, j);
                r0 += x < k0;
                r1 += x < k1;
            }
            for (uint32_t j = 32; j < n; ++j) {
                const uint32_t x = __shfl_sync(0xFFFFFFFFu, k1, j - 32u);
                r0 += x < k0;
                r1 += x < k1;
            }
#pragma unroll
            for (int q = 0; q < 2; ++q) {
                const uint32_t idx = q ? i1 : (uint32_t)lane;
                if (idx >= n) continue;
                const uint2 it = q ? it1 : it0;
                const uint32_t vid = a0 + (q ? r1 : r0);
                if (vid < fi.nvox) write_rank(p, fi.vbase + vid, f, vid, it.x, it.y);
                else {
                    set_status(p.hdr, MMBEV_DEV_BOUNDS);
                    zero_slot(p, it.x);
                }
            }
            continue;
        }
        for (int w = lane; w < nwords; w += 32) {
            bm_below[w] = 0u;
            if (capped) bm_tie[w] = 0u;
        }
        __syncwarp();
        for (uint32_t i = lane; i < n; i += 32) {
            const uint2 it = p.items[start + i];
            const uint32_t bit = it.y & lbmask;
            const bool tie = capped && slot_minrank(p, it.x) == fi.rstar;
            atomicOr(tie ? &bm_tie[bit >> 5] : &bm_below[bit >> 5], 1u << (bit & 31));
        }
        __syncwarp();
        // per-word exclusive prefix popcounts
        uint32_t sb = 0, st = 0;
        for (int k = 0; k < wpl; ++k) {
            const int w = lane * wpl + k;
            if (w < nwords) {
                sb += __popc(bm_below[w]);
                if (capped) st += __popc(bm_tie[w]);
            }
        }
        uint32_t ib = sb, it2 = st;
#pragma unroll
        for (int o2 = 1; o2 < 32; o2 <<= 1) {
            const uint32_t xb = __shfl_up_sync(0xFFFFFFFFu, ib, o2);
            const uint32_t xt = __shfl_up_sync(0xFFFFFFFFu, it2, o2);
            if (lane >= o2) { ib += xb; it2 += xt; }
        }
        uint32_t rb = ib - sb, rt = it2 - st;
        for (int k = 0; k < wpl; ++k) {
            const int w = lane * wpl + k;
            if (w < nwords) {
                pb[w] = (uint16_t)rb;
                rb += __popc(bm_below[w]);
                if (capped) {
                    pt[w] = (uint16_t)rt;
                    rt += __popc(bm_tie[w]);
                }
            }
        }
        __syncwarp();
        for (uint32_t i = lane; i < n; i += 32) {
            const uint2 it = p.items[start + i];
            const uint32_t h = it.x, lin = it.y;
            const uint32_t bit = lin & lbmask;
            const uint32_t w = bit >> 5, m = (1u << (bit & 31)) - 1u;
            const bool tie = capped && slot_minrank(p, h) == fi.rstar;
            const uint32_t A = a0 + pb[w] + __popc(bm_below[w] & m);
            const uint32_t c = capped ? c0 + pt[w] + __popc(bm_tie[w] & m) : 0u;
            bool kept;
            uint32_t vid;
            if (tie) { kept = c < fi.q; vid = A + c; }
            else { kept = true; vid = A + (c < fi.q ? c : fi.q); }
            if (kept && vid < fi.nvox) {
                write_rank(p, fi.vbase + vid, f, vid, h, lin);
            } else {
                if (kept) set_status(p.hdr, MMBEV_DEV_BOUNDS);
                zero_slot(p, h);  // dropped by the cap: release the slot
            }
        }
        __syncwarp();
    }
}

}  // namespace

cudaError_t launch_frames(const Params& p, int num_sms, bool pdl, cudaStream_t st) {
    return launch_k(k_frames, dim3(num_sms * 2), dim3(kThreads), 0, st, pdl, p);
}

cudaError_t launch_capped_census(const Params& p, int num_sms, bool pdl, cudaStream_t st) {
    return launch_k(k_capped_census, dim3(num_sms * 2), dim3(kThreads), 0, st, pdl, p);
}

cudaError_t launch_scan(const Params& p, bool pdl, cudaStream_t st) {
    return launch_k(k_scan, dim3(p.num_frames * p.scan_chunks), dim3(kScanThreads), 0, st, pdl,
                    p);
}

cudaError_t launch_scatter(const Params& p, int num_sms, bool pdl, cudaStream_t st) {
    return launch_k(k_scatter, dim3(num_sms * 4), dim3(kThreads), 0, st, pdl, p);
}

cudaError_t launch_rank(const Params& p, int num_sms, bool pdl, cudaStream_t st) {
    uint32_t blocks = (p.num_buckets + kRankWarps - 1) / kRankWarps;
    const uint32_t cap = (uint32_t)num_sms * 8u;
    if (blocks > cap) blocks = cap;
    if (blocks == 0) blocks = 1;
    return launch_k(k_rank, dim3(blocks), dim3(kRankWarps * 32), 0, st, pdl, p);
}

}  // namespace mmbev
