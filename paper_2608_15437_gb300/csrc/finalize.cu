// Stage 10: voxel feature encoder (S5 of the path; Alg. 1 "VoxelFeatureEncoder").
//
// Each kept voxel's slot gives its point count n and the start of its
// segment in `seg`, which lists the record positions of all n points (in
// arrival order). Record positions grow with the point index, so the voxel's
// first K points by index are its K smallest positions. The records (32
// bytes each, one sector) hold the compensated x', y', z' computed once by
// the classify pass with the Eq. 6 operation order, the intensity and dt.
// The five features are summed over the kept points in index order in fp32
// and divided once by the count; the feature row and the count are written
// and the slot is returned to the all-zero state.
//
// One launch, two roles. Light blocks: one thread per kept voxel with at
// most 32 points keeps the K smallest positions in a sorted register array
// (each position bubbles in with compare-and-swap steps; eight positions load
// at a time); the others are skipped. Heavy blocks (the first block indices,
// so they are dispatched first), over the slots the compact stage listed: one
// warp per voxel with 33 to 1024 points, where each lane keeps the smallest
// positions of its share of the segment, then K rounds of a warp minimum
// pick the voxel's K smallest in ascending order, the lanes fetch those
// records in parallel and lane 0 adds them up in order; a whole block per
// voxel with more than 1024 points (eight warps' lists merged by one). The
// heavy voxels' work so overlaps the light voxels'.
#include "mmbev_internal.cuh"

namespace mmbev {
namespace {

constexpr int kThreads = 256;

// Insert v into the ascending array b[0..B) (unused entries hold ~0u); the
// largest entry falls off the end.
template <int B>
__device__ __forceinline__ void sorted_insert(uint32_t (&b)[B], uint32_t v) {
#pragma unroll
    for (int j = 0; j < B; ++j) {
        const uint32_t lo = v < b[j] ? v : b[j];
        const uint32_t hi = v < b[j] ? b[j] : v;
        b[j] = lo;
        v = hi;
    }
}

// record: {x', y', z', intensity} {dt, rank, -, -}
__device__ __forceinline__ void add_record(float (&acc)[5], const uint4& a, float dt) {
    acc[0] = __fadd_rn(acc[0], __uint_as_float(a.x));
    acc[1] = __fadd_rn(acc[1], __uint_as_float(a.y));
    acc[2] = __fadd_rn(acc[2], __uint_as_float(a.z));
    acc[3] = __fadd_rn(acc[3], __uint_as_float(a.w));
    acc[4] = __fadd_rn(acc[4], dt);
}

// Load the features of the record at position q (clamped into the array).
__device__ __forceinline__ void load_record(const Params& p, uint32_t q, uint4& a, float& dt) {
    const uint4* rec = p.records + 2 * (size_t)min(q, p.rec_cap - 1u);
    a = __ldg(rec);
    dt = __ldg(reinterpret_cast<const float*>(rec + 1));
}

__device__ __forceinline__ void write_voxel(const Params& p, size_t row, const float (&acc)[5],
                                            int cnt) {
    const float fc = (float)cnt;
#pragma unroll
    for (int c = 0; c < 5; ++c) p.out_feats[row * 5 + c] = __fdiv_rn(acc[c], fc);
    p.out_counts[row] = cnt;
}

// Frame and output row of kept voxel g (s_vbase: prefix of kept voxels).
__device__ __forceinline__ size_t voxel_row(const Params& p, const uint32_t* s_vbase, int F,
                                            uint32_t g) {
    int lo = 0, hi = F;  // s_vbase[lo] <= g < s_vbase[hi]
    while (hi - lo > 1) {
        const int mid = (lo + hi) >> 1;
        if (s_vbase[mid] <= g) lo = mid; else hi = mid;
    }
    return (size_t)lo * (uint32_t)p.max_voxels + (g - s_vbase[lo]);
}

// Light role: block lb of nlb.
template <int B>
__device__ __forceinline__ void finalize_light(const Params& p, const uint32_t* s_vbase, int F,
                                               uint32_t total, uint32_t seg_cap, uint32_t lb,
                                               uint32_t nlb) {
    const uint32_t gs = nlb * blockDim.x;
    const int K = p.K;
    for (uint32_t g0 = lb * blockDim.x; g0 < total; g0 += gs) {
        const uint32_t g = g0 + threadIdx.x;
        const bool act = g < total;
        uint32_t h = 0, n = 0, off = 0;
        if (act) {
            h = p.vid_slot[g];
            const uint2 s = __ldcg(reinterpret_cast<const uint2*>(slot_key(p, h)));  // seg, -
            off = s.x;
            n = ld_cg(slot_cnt(p, h));
            if (off > seg_cap || n > seg_cap - off) {   // inconsistent lists: report, read nothing
                set_status(p.hdr, MMBEV_DEV_BOUNDS);
                n = 0;
            }
        }
        // heavy and huge voxels are the heavy role's; a count of 0 is a slot
        // that role has already returned to zero (a kept voxel has a point)
        if (!act || n == 0 || n > kLightMax) continue;
        uint32_t best[B];
#pragma unroll
        for (int j = 0; j < B; ++j) best[j] = 0xFFFFFFFFu;
        // the segment's positions, eight loads in flight at a time
        for (uint32_t i = 0; i < n; i += 8) {
            uint32_t v[8];
#pragma unroll
            for (int c = 0; c < 8; ++c) v[c] = i + c < n ? __ldg(p.seg + off + i + c) : 0xFFFFFFFFu;
#pragma unroll
            for (int c = 0; c < 8; ++c) sorted_insert<B>(best, v[c]);
        }
        const int cnt = (int)(n < (uint32_t)K ? n : (uint32_t)K);
        // the kept records, all loads of a round in flight, summed in order
        // (constant indices into `best` keep it in registers)
        constexpr int R = B < 3 ? B : 3;
        float acc[5] = {0.f, 0.f, 0.f, 0.f, 0.f};
#pragma unroll
        for (int j0 = 0; j0 < B; j0 += R) {
            if (j0 >= cnt) break;
            uint4 ra[R];
            float dt[R];
#pragma unroll
            for (int c = 0; c < R; ++c)
                if (j0 + c < cnt) {
                    if (best[j0 + c] >= p.rec_cap) set_status(p.hdr, MMBEV_DEV_BOUNDS);
                    load_record(p, best[j0 + c], ra[c], dt[c]);
                }
#pragma unroll
            for (int c = 0; c < R; ++c)
                if (j0 + c < cnt) add_record(acc, ra[c], dt[c]);
        }
        write_voxel(p, voxel_row(p, s_vbase, F, g), acc, cnt);
        zero_slot(p, h);
    }
}

// The j-th of a warp's cnt smallest positions sits in lane j % 32 (register
// j / 32): the lanes load those records in parallel and every lane adds them
// up in order (lane 0's sum is the one written).
__device__ __forceinline__ void warp_sum_records(const Params& p, const uint32_t (&mine)[2],
                                                 int cnt, int lane, float (&acc)[5]) {
    for (int half = 0; half * 32 < cnt; ++half) {
        uint4 ra = make_uint4(0u, 0u, 0u, 0u);
        float rdt = 0.f;
        if (half * 32 + lane < cnt) {
            if (mine[half] >= p.rec_cap) set_status(p.hdr, MMBEV_DEV_BOUNDS);
            load_record(p, mine[half], ra, rdt);
        }
        const int m = cnt - half * 32 < 32 ? cnt - half * 32 : 32;
        for (int j = 0; j < m; ++j) {
            uint4 a;
            a.x = __shfl_sync(0xFFFFFFFFu, ra.x, j);
            a.y = __shfl_sync(0xFFFFFFFFu, ra.y, j);
            a.z = __shfl_sync(0xFFFFFFFFu, ra.z, j);
            a.w = __shfl_sync(0xFFFFFFFFu, ra.w, j);
            add_record(acc, a, __shfl_sync(0xFFFFFFFFu, rdt, j));
        }
    }
}

// Heavy role: block hb of nhb (block-uniform, so its barriers are safe), over
// the slots the compact stage listed; the rank stage left each kept voxel's
// output index in its slot, and a listed slot the cap dropped is all-zero.
template <int B>
__device__ __forceinline__ void finalize_heavy(const Params& p, const uint32_t* s_vbase, int F,
                                               uint32_t total, uint32_t seg_cap, uint32_t hb,
                                               uint32_t nhb, uint32_t (*s_cand)[kMaxK]) {
    const int lane = threadIdx.x & 31;
    const int K = p.K;
    // Huge voxels, one block each: every thread keeps the smallest positions
    // of its share, each warp reduces its threads' to its K smallest, and
    // warp 0 merges the warps' lists.
    const uint32_t nhuge = ld_cg(&p.hdr->num_huge);
    const int warp = threadIdx.x >> 5;
    for (uint32_t e = hb; e < nhuge; e += nhb) {
        const uint32_t h = p.huge[e];
        const uint32_t off = ld_cg(slot_seg(p, h));
        uint32_t n = ld_cg(slot_cnt(p, h));
        if (n == 0) continue;   // dropped by the cap (the same for the whole block)
        const uint32_t g = ld_cg(slot_rank(p, h));
        if (g >= total) {
            if (threadIdx.x == 0) set_status(p.hdr, MMBEV_DEV_BOUNDS);
            continue;
        }
        if (off > seg_cap || n > seg_cap - off) {
            if (threadIdx.x == 0) set_status(p.hdr, MMBEV_DEV_BOUNDS);
            n = 0;
        }
        const int cnt = (int)(n < (uint32_t)K ? n : (uint32_t)K);
        uint32_t best[B];
#pragma unroll
        for (int j = 0; j < B; ++j) best[j] = 0xFFFFFFFFu;
        for (uint32_t i0 = threadIdx.x; i0 < n; i0 += 8u * kThreads) {
            uint32_t v[8];
#pragma unroll
            for (int c = 0; c < 8; ++c) {
                const uint32_t i = i0 + (uint32_t)kThreads * c;
                v[c] = i < n ? __ldg(p.seg + off + i) : 0xFFFFFFFFu;
            }
#pragma unroll
            for (int c = 0; c < 8; ++c) sorted_insert<B>(best, v[c]);
        }
        for (int j = 0; j < cnt; ++j) {
            const uint32_t m = __reduce_min_sync(0xFFFFFFFFu, best[0]);
            if (lane == 0) s_cand[warp][j] = m;
            if (best[0] == m) {
#pragma unroll
                for (int c = 0; c + 1 < B; ++c) best[c] = best[c + 1];
                best[B - 1] = 0xFFFFFFFFu;
            }
        }
        __syncthreads();
        if (warp == 0) {
#pragma unroll
            for (int j = 0; j < B; ++j) best[j] = 0xFFFFFFFFu;
            for (int i = lane; i < (kThreads / 32) * cnt; i += 32)
                sorted_insert<B>(best, s_cand[i / cnt][i % cnt]);
            uint32_t mine[2] = {0xFFFFFFFFu, 0xFFFFFFFFu};
            for (int j = 0; j < cnt; ++j) {
                const uint32_t m = __reduce_min_sync(0xFFFFFFFFu, best[0]);
                if (lane == (j & 31)) mine[j >> 5] = m;
                if (best[0] == m) {
#pragma unroll
                    for (int c = 0; c + 1 < B; ++c) best[c] = best[c + 1];
                    best[B - 1] = 0xFFFFFFFFu;
                }
            }
            float acc[5] = {0.f, 0.f, 0.f, 0.f, 0.f};
            warp_sum_records(p, mine, cnt, lane, acc);
            if (lane == 0) {
                write_voxel(p, voxel_row(p, s_vbase, F, g), acc, cnt);
                zero_slot(p, h);
            }
        }
        __syncthreads();
    }
    const uint32_t nh = ld_cg(&p.hdr->num_heavy);
    const uint32_t gw = (hb * blockDim.x + threadIdx.x) >> 5;
    const uint32_t nw = (nhb * blockDim.x) >> 5;
    for (uint32_t e = gw; e < nh; e += nw) {
        const uint32_t h = p.heavy[e];
        const uint32_t off = ld_cg(slot_seg(p, h));
        uint32_t n = ld_cg(slot_cnt(p, h));
        if (n == 0) continue;   // dropped by the cap (the same for the whole warp)
        const uint32_t g = ld_cg(slot_rank(p, h));
        if (g >= total) {
            if (lane == 0) set_status(p.hdr, MMBEV_DEV_BOUNDS);
            continue;
        }
        if (off > seg_cap || n > seg_cap - off) {   // inconsistent lists: report, read nothing
            if (lane == 0) set_status(p.hdr, MMBEV_DEV_BOUNDS);
            n = 0;
        }
        uint32_t best[B];
#pragma unroll
        for (int j = 0; j < B; ++j) best[j] = 0xFFFFFFFFu;
        // each lane takes every 32nd position, eight loads in flight at a time
        for (uint32_t i0 = lane; i0 < n; i0 += 256) {
            uint32_t v[8];
#pragma unroll
            for (int c = 0; c < 8; ++c) {
                const uint32_t i = i0 + 32u * c;
                v[c] = i < n ? __ldg(p.seg + off + i) : 0xFFFFFFFFu;
            }
#pragma unroll
            for (int c = 0; c < 8; ++c) sorted_insert<B>(best, v[c]);
        }
        // K rounds of a warp minimum over the lanes' smallest remaining; the
        // j-th smallest goes to lane j % 32 (second register for j >= 32)
        const int cnt = (int)(n < (uint32_t)K ? n : (uint32_t)K);
        uint32_t mine[2] = {0xFFFFFFFFu, 0xFFFFFFFFu};
        for (int j = 0; j < cnt; ++j) {
            const uint32_t m = __reduce_min_sync(0xFFFFFFFFu, best[0]);
            if (lane == (j & 31)) mine[j >> 5] = m;
            if (best[0] == m) {   // positions are distinct: one lane owns m
#pragma unroll
                for (int c = 0; c + 1 < B; ++c) best[c] = best[c + 1];
                best[B - 1] = 0xFFFFFFFFu;
            }
        }
        float acc[5] = {0.f, 0.f, 0.f, 0.f, 0.f};
        warp_sum_records(p, mine, cnt, lane, acc);
        if (lane == 0) {
            write_voxel(p, voxel_row(p, s_vbase, F, g), acc, cnt);
            zero_slot(p, h);
        }
    }
}

// Up to K = 12, six blocks fit an SM (40 registers, no spill): the light
// blocks start beside the heavy ones.
template <int BL, int BH>
__global__ void __launch_bounds__(kThreads, (BL <= 12 ? 6 : 1))
    k_finalize(Params p, uint32_t heavy_blocks) {
    __shared__ uint32_t s_vbase[kMaxFrames + 1];
    __shared__ uint32_t s_cand[kThreads / 32][kMaxK];
    pdl_wait();
    const int F = p.num_frames;
    for (int i = threadIdx.x; i < F; i += blockDim.x) s_vbase[i] = p.finfo[i].vbase;
    const uint32_t total = ld_cg(&p.hdr->total_kept);
    const uint32_t seg_cap = min(ld_cg(&p.hdr->seg_total), p.occ_cap);  // seg holds N entries
    if (threadIdx.x == 0) s_vbase[F] = total;
    __syncthreads();
    if (blockIdx.x < heavy_blocks)
        finalize_heavy<BH>(p, s_vbase, F, total, seg_cap, blockIdx.x, heavy_blocks, s_cand);
    else
        finalize_light<BL>(p, s_vbase, F, total, seg_cap, blockIdx.x - heavy_blocks,
                           gridDim.x - heavy_blocks);
}

}  // namespace

cudaError_t launch_finalize(const Params& p, int num_sms, bool pdl, cudaStream_t st) {
    // two heavy blocks per SM, six light ones, so the light blocks start
    // while the heavy ones run
    const uint32_t heavy = (uint32_t)num_sms * 2;
    const dim3 grid(num_sms * 8), block(kThreads);
    if (p.K <= 4) return launch_k(k_finalize<4, 4>, grid, block, 0, st, pdl, p, heavy);
    if (p.K <= 12) return launch_k(k_finalize<12, 12>, grid, block, 0, st, pdl, p, heavy);
    if (p.K <= 32) return launch_k(k_finalize<32, 32>, grid, block, 0, st, pdl, p, heavy);
    return launch_k(k_finalize<32, kMaxK>, grid, block, 0, st, pdl, p, heavy);
}

}  // namespace mmbev
