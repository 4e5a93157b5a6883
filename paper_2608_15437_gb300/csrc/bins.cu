// Stages 2-6: voxel dedup (S3), cap and canonical order (S4), first-K mean
// features (S5) of the path (Alg. 1 "Voxelize" and "VoxelFeatureEncoder";
// Sec. IV-F hard voxelization; Sec. IV-C mandatory ROIs first).
//
// The classify pass has counted every kept point into its bucket (2^LB
// consecutive linear indices of one frame; bucket b = frame * Bf + lin >> LB,
// so buckets ascend with (frame, lin)). Then:
//
//   scan     (stage 2)  exclusive prefix of the bucket counts over the whole
//                       call (one pass, tiles of 4,096 buckets chained by
//                       decoupled look-back: a tile publishes its total, then
//                       its inclusive prefix once its predecessors' are
//                       known), and the non-empty buckets listed as warp jobs
//                       (at most 256 points), block jobs (at most 2,048) or
//                       parts of 2,048 points of a larger bucket.
//   scatter  (stage 3)  a counting sort of the kept points by bucket: entry
//                       {position, low lin bits | rank} goes to item
//                       boff[bucket] + its arrival, numbered by one atomic
//                       per group of a warp's entries that share a bucket.
//   buckets  (stage 4)  each bucket (or part) alone: its voxels are the
//                       distinct low lin bits of its points, ranked by an
//                       occupancy bitmap (popcount prefix), so voxel v of the
//                       bucket is the v-th smallest lin; a counting sort by
//                       voxel gives each voxel its points, and of those the K
//                       smallest record positions (= smallest point indices)
//                       are written in ascending order to vitems, with the
//                       voxel's descriptor {first vitem, point count, low lin
//                       bits, minimum rank} at vdesc[boff + v]. A warp takes a
//                       bucket of up to 32 points in registers and one of up
//                       to 256 in shared memory, a block a larger one or a
//                       part. The bucket's voxel count goes to ucnt and to its
//                       frame slice's sum.
//   merge    (stage 5)  a block per bucket split in parts combines the parts'
//                       voxels: counts add, minimum ranks take the minimum,
//                       and the K smallest of the parts' kept positions are
//                       the voxel's.
//   output   (stage 6)  per frame slice of 512 buckets: the slice sums and a
//                       scan of the bucket counts give every voxel its output
//                       row (ascending lin); a lane per voxel sums the
//                       records of its kept points in index order in fp32,
//                       divides once and writes the row. A frame over
//                       max_voxels keeps the max_voxels smallest by (minimum
//                       rank, lin): a histogram of minimum ranks gives the
//                       threshold rank r* and the quota q of rank-r* voxels
//                       that fit; rank-r* voxels are kept in ascending lin
//                       until q are taken.
#include <atomic>

#include "mmbev_internal.cuh"

namespace mmbev {
namespace {

constexpr uint32_t kFull = 0xFFFFFFFFu;

// ------------------------------------------------------------------ helpers

// Exclusive scan of one value per thread over the block; total in *total.
// s_warp holds blockDim/32 words. Every thread must call it (two barriers).
__device__ __forceinline__ uint32_t block_exclusive_scan(uint32_t v, uint32_t* s_warp,
                                                         uint32_t* total) {
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int nwarps = (int)(blockDim.x >> 5);
    uint32_t inc = v;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        const uint32_t x = __shfl_up_sync(kFull, inc, o);
        if (lane >= o) inc += x;
    }
    if (lane == 31) s_warp[warp] = inc;
    __syncthreads();
    uint32_t wbase = 0, tot = 0;
    for (int w = 0; w < nwarps; ++w) {
        const uint32_t x = s_warp[w];
        if (w < warp) wbase += x;
        tot += x;
    }
    __syncthreads();
    *total = tot;
    return wbase + inc - v;
}

__device__ __forceinline__ uint32_t warp_exclusive_scan(uint32_t v, uint32_t* total) {
    const int lane = threadIdx.x & 31;
    uint32_t inc = v;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        const uint32_t x = __shfl_up_sync(kFull, inc, o);
        if (lane >= o) inc += x;
    }
    *total = __shfl_sync(kFull, inc, 31);
    return inc - v;
}

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

// Ascending order of a[0..B) (unused entries ~0u, which end last): an
// odd-even transposition network for small B, a bitonic network for the
// larger (power-of-two) ones.
template <int B>
__device__ __forceinline__ void sort_small(uint32_t (&a)[B]) {
    if constexpr (B <= 16) {
#pragma unroll
        for (int r = 0; r < B; ++r)
#pragma unroll
            for (int j = r & 1; j + 1 < B; j += 2) {
                const uint32_t lo = min(a[j], a[j + 1]), hi = max(a[j], a[j + 1]);
                a[j] = lo;
                a[j + 1] = hi;
            }
    } else {
        static_assert((B & (B - 1)) == 0, "bitonic network: a power of two");
#pragma unroll
        for (int k = 2; k <= B; k <<= 1)
#pragma unroll
            for (int j = k >> 1; j > 0; j >>= 1)
#pragma unroll
                for (int i = 0; i < B; ++i) {
                    const int l = i ^ j;
                    if (l > i) {
                        const uint32_t lo = min(a[i], a[l]), hi = max(a[i], a[l]);
                        const bool up = (i & k) == 0;
                        a[i] = up ? lo : hi;
                        a[l] = up ? hi : lo;
                    }
                }
    }
}

// Low lin bits of an item's second word, masked to the bucket's size: an
// index into a bucket bitmap whatever the word holds.
__device__ __forceinline__ uint32_t item_lo(const Params& p, uint32_t y) {
    return y & ((1u << p.bucket_log2) - 1u);
}

// Voxel of low lin bits `lo` in a bucket: its rank among the bucket's
// distinct low bits, from the occupancy bitmap and its word prefixes.
__device__ __forceinline__ uint32_t voxel_of(const uint32_t* bm, const uint32_t* wpre, uint32_t lo) {
    const uint32_t w = lo >> 5;
    return wpre[w] + __popc(bm[w] & ((1u << (lo & 31)) - 1u));
}

// Output slices: a frame's buckets in groups of 2^kSliceLog2.
constexpr int kSliceLog2 = 9;

// The bucket's voxel count into ucnt, its frame slice's sum and its frame's
// total.
__device__ __forceinline__ void publish_bucket(const Params& p, uint32_t b, uint32_t nv) {
    p.ucnt[b] = nv;
    if (nv) {
        const uint32_t f = udiv(p.div_bf, b);
        const uint32_t bi = b - f * p.buckets_per_frame;
        atomicAdd(&p.ssum[f * p.out_slices + (bi >> kSliceLog2)], nv);
        atomicAdd(&p.ftot[f], nv);
    }
}

// Where a voxel's kept positions go: out[j * stride] for j < kept, and the
// index its descriptor records for them (`at`): vitems for a whole bucket,
// the .x words of the items array for one part of a bucket split in parts.
struct KeptOut {
    uint32_t* out;
    uint32_t stride;
    uint32_t at;
};

// Voxels of at most 32 points, a thread per point (entry i of a job's
// voxel-sorted entries). A voxel of at most K points keeps all its points:
// each goes to the voxel's kept list at its place in the voxel's run, in no
// particular order (the output stage sorts a voxel's kept positions before
// summing). In a denser one a point's rank by position among the voxel's
// points is where it goes, if below K. The voxel's first entry also writes
// the descriptor (count, low bits, minimum rank). Denser voxels are selected
// by a warp or by the block.
template <typename KO>
__device__ __forceinline__ void select_small(const Params& p, const uint2* seg, uint32_t i,
                                             const uint32_t* bm, const uint32_t* wpre,
                                             const uint32_t* vc, const KO& kept_out,
                                             uint4* desc) {
    const uint2 me = seg[i];
    const uint32_t lo = item_lo(p, me.y);
    const uint32_t v = voxel_of(bm, wpre, lo);
    const uint32_t st = v ? vc[v - 1] : 0u, cnt = vc[v] - st;
    if (cnt > 32u) return;
    const uint32_t K = (uint32_t)p.K;
    uint32_t r = i - st;
    if (cnt > K) {
        r = 0;
        for (uint32_t j = st; j < st + cnt; ++j) r += seg[j].x < me.x ? 1u : 0u;
    }
    const KeptOut ko = kept_out(st);
    if (r < K) ko.out[r * ko.stride] = me.x;
    if (i == st) {
        uint32_t mr = kUnset;
        for (uint32_t j = st; j < st + cnt; ++j) mr = min(mr, seg[j].y >> 16);
        desc[v] = make_uint4(ko.at, cnt, lo, mr);
    }
}

// One voxel by a whole warp (any count): each lane keeps the B smallest
// positions of every 32nd entry; K rounds of a warp minimum pick the K
// smallest in ascending order, and the lane that owns the j-th writes it.
template <int B>
__device__ __forceinline__ void select_by_warp(const Params& p, const uint2* seg, uint32_t st,
                                               uint32_t cnt, const KeptOut& ko, uint4* desc) {
    const int lane = threadIdx.x & 31;
    uint32_t best[B];
#pragma unroll
    for (int j = 0; j < B; ++j) best[j] = kUnset;
    uint32_t mr = kUnset;
    for (uint32_t i0 = lane; i0 < cnt; i0 += 32 * 4) {   // four entries in flight a lane
        uint2 e[4];
#pragma unroll
        for (int c = 0; c < 4; ++c) {
            const uint32_t i = i0 + 32u * c;
            e[c] = i < cnt ? seg[st + i] : make_uint2(kUnset, kUnset);
        }
#pragma unroll
        for (int c = 0; c < 4; ++c) {
            sorted_insert<B>(best, e[c].x);
            mr = min(mr, e[c].y >> 16);
        }
    }
    mr = __reduce_min_sync(kFull, mr);
    const uint32_t lo = item_lo(p, seg[st].y);
    const uint32_t kept = min(cnt, (uint32_t)p.K);
    for (uint32_t j = 0; j < kept; ++j) {
        const uint32_t m = __reduce_min_sync(kFull, best[0]);
        if (best[0] == m) {   // positions are distinct: one lane owns m
            ko.out[j * ko.stride] = m;
#pragma unroll
            for (int c = 0; c + 1 < B; ++c) best[c] = best[c + 1];
            best[B - 1] = kUnset;
        }
    }
    if (lane == 0) *desc = make_uint4(ko.at, cnt, lo, mr);
}

// Voxels of more than kWarpMax points are selected by a whole block (at
// most kHugeList a bucket; beyond that by warps).
constexpr uint32_t kWarpMax = 1024;
constexpr uint32_t kHugeList = 32;
// Voxels of 33 .. kWarpMax points a block job lists for its warps: a job of
// at most kPart points has at most kPart / 33 of them.
constexpr uint32_t kDenseList = 64;
static_assert(kPart / 33 < kDenseList, "a block job's dense voxels fit the list");

// One voxel by the whole block (every thread calls it): each thread keeps
// the B smallest positions of every blockDim-th entry, each warp reduces its
// lanes' to its K smallest in s_cand (blockDim/32 x B words of free shared
// memory), warp 0 merges those, and the lane owning the j-th smallest writes
// it.
template <int B>
__device__ __forceinline__ void select_by_block(const Params& p, const uint2* seg, uint32_t st,
                                                uint32_t cnt, const KeptOut& ko, uint4* desc,
                                                uint32_t* s_cand) {
    const int t = threadIdx.x, lane = t & 31, warp = t >> 5;
    const uint32_t nthr = blockDim.x;
    __shared__ uint32_t s_mr;
    if (t == 0) s_mr = kUnset;
    __syncthreads();
    uint32_t best[B];
#pragma unroll
    for (int j = 0; j < B; ++j) best[j] = kUnset;
    uint32_t mr = kUnset;
    for (uint32_t i0 = t; i0 < cnt; i0 += nthr * 4) {
        uint2 e[4];
#pragma unroll
        for (int c = 0; c < 4; ++c) {
            const uint32_t i = i0 + nthr * c;
            e[c] = i < cnt ? seg[st + i] : make_uint2(kUnset, kUnset);
        }
#pragma unroll
        for (int c = 0; c < 4; ++c) {
            sorted_insert<B>(best, e[c].x);
            mr = min(mr, e[c].y >> 16);
        }
    }
    const uint32_t kept = min(cnt, (uint32_t)p.K);
    for (uint32_t j = 0; j < kept; ++j) {
        const uint32_t m = __reduce_min_sync(kFull, best[0]);
        if (lane == 0) s_cand[warp * B + j] = m;
        if (best[0] == m) {
#pragma unroll
            for (int c = 0; c + 1 < B; ++c) best[c] = best[c + 1];
            best[B - 1] = kUnset;
        }
    }
    mr = __reduce_min_sync(kFull, mr);
    if (lane == 0) atomicMin(&s_mr, mr);
    __syncthreads();
    if (warp == 0) {
#pragma unroll
        for (int j = 0; j < B; ++j) best[j] = kUnset;
        const uint32_t nc = (nthr / 32) * kept;
        for (uint32_t i = lane; i < nc; i += 32) sorted_insert<B>(best, s_cand[(i / kept) * B + i % kept]);
        for (uint32_t j = 0; j < kept; ++j) {
            const uint32_t m = __reduce_min_sync(kFull, best[0]);
            if (best[0] == m) {
                ko.out[j * ko.stride] = m;
#pragma unroll
                for (int c = 0; c + 1 < B; ++c) best[c] = best[c + 1];
                best[B - 1] = kUnset;
            }
        }
        if (lane == 0) *desc = make_uint4(ko.at, cnt, item_lo(p, seg[st].y), s_mr);
    }
    __syncthreads();
}

// Insert position `pos` into the ascending K smallest ks[0..K) that many
// threads update at once (unused slots hold ~0u): each atomicMin leaves the
// smaller of the slot and the carried value in the slot and carries the
// larger on, so slot j ends as the (j+1)-th smallest of all inserted values
// whatever the interleaving; an empty slot ends the walk. Slots only shrink,
// so a slot read (even stale) below the carried value can be skipped.
// Returns false when pos cannot be among the K smallest.
__device__ __forceinline__ bool kmin_insert(uint32_t* ks, uint32_t K, uint32_t pos) {
    if (pos >= *reinterpret_cast<volatile uint32_t*>(&ks[K - 1])) return false;
    uint32_t v = pos;
    for (uint32_t j = 0; j < K; ++j) {
        if (*reinterpret_cast<volatile uint32_t*>(&ks[j]) < v) continue;
        const uint32_t old = atomicMin(&ks[j], v);
        if (old == kUnset) return true;
        if (old > v) v = old;
    }
    return true;
}

// Low lin bits of voxel v of a bucket: the v-th set bit of its occupancy
// bitmap (the last word whose prefix is <= v holds it).
__device__ __forceinline__ uint32_t lo_of_voxel(const uint32_t* bm, const uint32_t* wpre,
                                                uint32_t nwords, uint32_t v) {
    uint32_t a = 0, z = nwords;
    while (z - a > 1) {
        const uint32_t mid = (a + z) >> 1;
        if (wpre[mid] <= v) a = mid; else z = mid;
    }
    return a * 32u + __fns(bm[a], 0u, (int)(v - wpre[a] + 1u));
}

// ------------------------------------------------------------------ stage 2

constexpr int kScanThreads = 1024;
constexpr uint32_t kUnionWords = (1u << kBucketLog2Max) / 32;   // a split bucket's union bitmap
static_assert(kScanTile == kScanThreads * 4, "four buckets a thread");
constexpr unsigned long long kAggFlag = 1ull << 32;    // tile total published
constexpr unsigned long long kIncFlag = 2ull << 32;    // tile inclusive prefix published

// Size class of a block job (a bucket of kWarpJobMax+1 .. kPart points):
// 0 for 1,025-2,048 points, 1 for 513-1,024, 2 for 257-512; 3 otherwise.
__device__ __forceinline__ uint32_t block_job_class(uint32_t c) {
    if (c <= kWarpJobMax || c > kPart) return 3u;
    return c > kPart / 2 ? 0u : c > kPart / 4 ? 1u : 2u;
}

// Stage 2. The tile's inclusive prefix comes from its predecessors by
// decoupled look-back, done by warp 0 over 32 predecessors at a time: each
// lane waits (bounded) until its predecessor has published at least its
// total, and the nearest one that has published its inclusive prefix ends
// the walk. Then every non-empty bucket becomes jobs of the bucket stage: a
// small one (at most kWarpJobMax points) a warp job, a larger one a block job
// (in one of three size classes), and one of more than kPart points
// kPart-point parts, with the merge tasks that combine their voxel lists.
__global__ void __launch_bounds__(kScanThreads) k_bucket_scan(Params p) {
    __shared__ uint32_t s_warp[kScanThreads / 32];
    __shared__ uint32_t s_tile, s_base, s_jbase[4];
    pdl_wait();
    const int t = threadIdx.x, lane = t & 31;
    // tiles are numbered in the order their blocks start, so a tile only
    // ever waits on tiles whose blocks are already running
    if (t == 0) s_tile = atomicAdd(&p.hdr->scan_ticket, 1u);
    __syncthreads();
    const uint32_t tile = s_tile;
    if (tile >= p.scan_tiles) return;
    const uint32_t B = p.num_buckets;
    const uint32_t b0 = tile * kScanTile + 4u * (uint32_t)t;
    uint32_t c[4], sum = 0;
#pragma unroll
    for (int k = 0; k < 4; ++k) {
        c[k] = b0 + k < B ? p.bcnt[b0 + k] : 0u;
        sum += c[k];
    }
    uint32_t total = 0;
    const uint32_t excl = block_exclusive_scan(sum, s_warp, &total);
    if (t < 32) {
        unsigned long long* st = p.scan_state;
        uint32_t base = 0;
        if (tile == 0) {
            if (lane == 0) atomicExch(&st[0], kIncFlag | total);
        } else {
            if (lane == 0) atomicExch(&st[tile], kAggFlag | total);
            int64_t j = (int64_t)tile - 1;
            for (;;) {
                const int64_t q = j - lane;
                unsigned long long w = kIncFlag;   // before tile 0: an inclusive prefix of 0
                bool gave_up = false;
                if (q >= 0) {
                    uint32_t spins = 0;
                    while (((w = ld_acquire(&st[q])) >> 32) == 0ull) {
                        if (++spins >= kSpinLimit) {
                            gave_up = true;
                            break;
                        }
                    }
                }
                if (__any_sync(kFull, gave_up)) {   // the results are void
                    if (lane == 0) set_status(p.hdr, MMBEV_DEV_WAIT_TIMEOUT);
                    break;
                }
                const uint32_t inc = __ballot_sync(kFull, (w & kIncFlag) != 0ull);
                const int last = inc ? __ffs(inc) - 1 : 31;   // lanes 0..last contribute
                uint32_t v = lane <= last ? (uint32_t)w : 0u;
#pragma unroll
                for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(kFull, v, o);
                base += v;
                if (inc) break;
                j -= 32;
            }
            if (lane == 0) atomicExch(&st[tile], kIncFlag | (unsigned long long)(base + total));
        }
        if (lane == 0) s_base = base;
    }
    __syncthreads();
    // the tile's warp jobs and block jobs (three size classes, so that the
    // bucket stage takes the largest first): one reservation a list for the
    // whole tile (counts packed two to a word; a tile has 4,096 buckets)
    uint32_t jc0 = 0, jc1 = 0;
#pragma unroll
    for (int k = 0; k < 4; ++k) {
        const bool ok = b0 + k < B;
        const uint32_t cls = block_job_class(c[k]);
        jc0 += ok && c[k] > 0u && c[k] <= kWarpJobMax ? 1u : 0u;
        jc0 += ok && cls == 0u ? 1u << 16 : 0u;
        jc1 += ok && cls == 1u ? 1u : 0u;
        jc1 += ok && cls == 2u ? 1u << 16 : 0u;
    }
    uint32_t jt0 = 0, jt1 = 0;
    const uint32_t je0 = block_exclusive_scan(jc0, s_warp, &jt0);
    const uint32_t je1 = block_exclusive_scan(jc1, s_warp, &jt1);
    if (t == 0) {
        const uint32_t ns0 = jt0 & 0xFFFFu, nl0 = jt0 >> 16, nl1 = jt1 & 0xFFFFu, nl2 = jt1 >> 16;
        s_jbase[0] = ns0 ? atomicAdd(&p.hdr->n_small, ns0) : 0u;
        s_jbase[1] = nl0 ? atomicAdd(&p.hdr->n_large[0], nl0) : 0u;
        s_jbase[2] = nl1 ? atomicAdd(&p.hdr->n_large[1], nl1) : 0u;
        s_jbase[3] = nl2 ? atomicAdd(&p.hdr->n_large[2], nl2) : 0u;
    }
    __syncthreads();
    uint32_t js = s_jbase[0] + (je0 & 0xFFFFu);
    uint32_t jl0 = s_jbase[1] + (je0 >> 16), jl1 = s_jbase[2] + (je1 & 0xFFFFu),
             jl2 = s_jbase[3] + (je1 >> 16);
    uint32_t run = s_base + excl;
#pragma unroll
    for (int k = 0; k < 4; ++k) {
        const uint32_t b = b0 + k;
        if (b < B) {
            p.boff[b] = run;
            p.ucnt[b] = 0u;
            if (b == B - 1u) p.boff[B] = run + c[k];
        }
        const uint4 d = make_uint4(b, run, c[k], kUnset);
        if (b < B && c[k] > 0u && c[k] <= kWarpJobMax) {
            if (js < B) p.sjobs[js] = d;
            else set_status(p.hdr, MMBEV_DEV_BOUNDS);
            ++js;
        }
        const uint32_t cls = block_job_class(c[k]);
        if (b < B && cls < 3u) {
            const uint32_t at = cls == 0u ? jl0++ : cls == 1u ? jl1++ : jl2++;
            if (at < p.job_cap) p.jobs[(size_t)cls * p.job_cap + at] = d;
            else set_status(p.hdr, MMBEV_DEV_BOUNDS);
        }
        if (b < B && c[k] > kPart) {   // parts of a bucket too large for one block
            const uint32_t P = (c[k] + kPart - 1) / kPart;
            const uint32_t h = atomicAdd(&p.hdr->n_huge, 1u);
            const uint32_t j0 = atomicAdd(&p.hdr->n_parts, P);
            if (h < p.huge_cap && j0 + P <= p.part_cap) {
                p.hj0[h] = j0;
                uint4* hb = reinterpret_cast<uint4*>(p.hbits + (size_t)h * kUnionWords);
                for (uint32_t w = 0; w < kUnionWords / 4; ++w) hb[w] = make_uint4(0u, 0u, 0u, 0u);
                for (uint32_t q = 0; q < P; ++q)
                    p.hjobs[j0 + q] = make_uint4(b, run + q * kPart, min(kPart, c[k] - q * kPart), h);
                // merge tasks: W ranges of the bitmap words, one per kMergeItems points
                const uint32_t nwords = (1u << p.bucket_log2) >= 32u ? (1u << p.bucket_log2) >> 5 : 1u;
                const uint32_t W = min((c[k] + kMergeItems - 1) / kMergeItems, nwords);
                const uint32_t m0 = atomicAdd(&p.hdr->n_mtasks, W);
                if (m0 + W <= p.mtask_cap) {
                    for (uint32_t w = 0; w < W; ++w) p.mtasks[m0 + w] = make_uint2(h, w | W << 16);
                } else {
                    set_status(p.hdr, MMBEV_DEV_BOUNDS);
                }
            } else {
                set_status(p.hdr, MMBEV_DEV_BOUNDS);
            }
        }
        run += c[k];
    }
}

// ------------------------------------------------------------------ stage 3

constexpr int kThreads = 256;

// Prefix sums of the classify blocks' list lengths (off[0..G]) and of their
// units of kUnit entries (uoff[0..G]), and the first plist entry of each list
// (list l starts at tile t_begin(l) * 2048).
constexpr uint32_t kUnit = 128;   // entries a warp takes at once (4 per lane)
struct Lists {
    uint32_t off[kMaxClsGrid + 1];
    uint32_t uoff[kMaxClsGrid + 1];
    uint32_t start[kMaxClsGrid];
};

// Every thread must call it (two barriers). Returns the entry count.
__device__ __forceinline__ uint32_t lists_scan(const Params& p, Lists& L, uint32_t* s_warp) {
    const uint32_t G = p.cls_grid;
    const uint64_t T = (uint64_t)p.num_regions / (kTile / kRegion);
    // kMaxClsGrid <= kThreads * 4: each thread scans up to 4 consecutive lists
    uint32_t c[4], sum = 0;
#pragma unroll
    for (int k = 0; k < 4; ++k) {
        const uint32_t l = (uint32_t)threadIdx.x * 4 + k;
        c[k] = 0;
        if (l < G) {
            const uint64_t t0 = (uint64_t)l * T / G;
            const uint64_t room = ((uint64_t)(l + 1) * T / G - t0) * kTile;
            c[k] = (uint32_t)min((uint64_t)p.cls_cnt[l], room);
            L.start[l] = (uint32_t)(t0 * kTile);
        }
        sum += c[k];
    }
    uint32_t usum = 0;
#pragma unroll
    for (int k = 0; k < 4; ++k) usum += (c[k] + kUnit - 1) / kUnit;
    uint32_t total = 0, utotal = 0;
    uint32_t run = block_exclusive_scan(sum, s_warp, &total);
    uint32_t urun = block_exclusive_scan(usum, s_warp, &utotal);
#pragma unroll
    for (int k = 0; k < 4; ++k) {
        const uint32_t l = (uint32_t)threadIdx.x * 4 + k;
        if (l <= G) {
            L.off[l] = run;
            L.uoff[l] = urun;
        }
        run += c[k];
        urun += (c[k] + kUnit - 1) / kUnit;
    }
    __syncthreads();
    return L.uoff[G];
}

// Each warp takes units of kUnit consecutive entries of one classify block's
// list (four groups of 32); eight blocks an SM, for twice the loads and
// atomics in flight that 32 registers a thread allow. The entries of one bucket in a group take their
// places with one atomic on the bucket's cursor (ucnt, zero after the scan
// stage; it ends at the bucket's count).
__global__ void __launch_bounds__(kThreads, 8) k_bucket_scatter(Params p) {
    __shared__ Lists L;
    __shared__ uint32_t s_warp[kThreads / 32];
    pdl_wait();
    const uint32_t NU = lists_scan(p, L, s_warp);
    const uint32_t G = p.cls_grid;
    const int lane = threadIdx.x & 31;
    const uint32_t lt = (1u << lane) - 1u;
    const uint32_t gw = (blockIdx.x * blockDim.x + threadIdx.x) >> 5;
    const uint32_t nw = (gridDim.x * blockDim.x) >> 5;
    constexpr int U = kUnit / 32;
    for (uint32_t unit = gw; unit < NU; unit += nw) {   // warp-uniform
        uint32_t l = 0, hi = G;   // its list: uoff[l] <= unit < uoff[l + 1]
        while (hi - l > 1) {
            const uint32_t mid = (l + hi) >> 1;
            if (L.uoff[mid] <= unit) l = mid; else hi = mid;
        }
        const uint32_t k0 = (unit - L.uoff[l]) * kUnit, cnt = L.off[l + 1] - L.off[l];
        const uint4* src = p.plist + L.start[l];
        uint4 e[U];
#pragma unroll
        for (int u = 0; u < U; ++u) {
            const uint32_t j = k0 + (uint32_t)u * 32u + (uint32_t)lane;
            e[u] = j < cnt ? __ldcs(src + j) : make_uint4(kUnset, 0u, 0u, 0u);
            if (e[u].x >= p.num_buckets) e[u].x = kUnset;
        }
        // The entries of one bucket in a group of 32 take their arrival
        // numbers with one atomic by the group's first lane. Every number and
        // bucket offset is requested before any is used, so that their
        // latencies overlap.
        uint32_t bo[U], grp[U], old[U];
#pragma unroll
        for (int u = 0; u < U; ++u) bo[u] = e[u].x != kUnset ? __ldg(p.boff + e[u].x) : 0u;
#pragma unroll
        for (int u = 0; u < U; ++u) grp[u] = __match_any_sync(kFull, e[u].x);
#pragma unroll
        for (int u = 0; u < U; ++u) {
            old[u] = 0u;
            if (e[u].x != kUnset && lane == __ffs(grp[u]) - 1)
                old[u] = atomicAdd(&p.ucnt[e[u].x], (uint32_t)__popc(grp[u]));
        }
#pragma unroll
        for (int u = 0; u < U; ++u)
            old[u] = __shfl_sync(kFull, old[u], __ffs(grp[u]) - 1) + __popc(grp[u] & lt);
#pragma unroll
        for (int u = 0; u < U; ++u) {
            if (e[u].x == kUnset) continue;
            const uint32_t at = bo[u] + old[u];
            if (at < p.item_cap) p.items[at] = make_uint2(e[u].y, e[u].z);
            else set_status(p.hdr, MMBEV_DEV_BOUNDS);
        }
    }
}

// ------------------------------------------------------------------ stage 4

// Bucket-stage blocks: 128 threads. A block job (more than kWarpJobMax and
// at most kPart points) uses the whole block; a warp job (at most
// kWarpJobMax points) one warp, in its own piece of the block's shared
// memory.
constexpr int kBT = 128;
constexpr int kBmWords = (1 << kBucketLog2Max) / 32;    // 256
constexpr size_t kBlockSmem = (size_t)kBmWords * 4 * 2 + (size_t)kPart * 4 +
                              (size_t)kPart * sizeof(uint2);
constexpr size_t kWarpSmem = (size_t)kBmWords * 4 * 2 + kWarpJobMax * 4 + kWarpJobMax * sizeof(uint2);
static_assert(kWarpSmem * (kBT / 32) <= kBlockSmem, "the warp pieces fit");
constexpr uint32_t kIl = 4;   // items a thread keeps in registers: jobs up to 512 points

// A block job (more than kWarpJobMax and at most kPart points): a whole
// bucket, or part of a bucket split in parts (then job.w is the split
// bucket's index). job = {bucket, first item, points, split index or ~0};
// jidx its place in the job list.
template <int BH>
__device__ void bucket_by_block(const Params& p, const uint4& job, uint32_t jidx,
                                unsigned char* smem, uint32_t* s_warp) {
    const int t = threadIdx.x, warp = t >> 5;
    uint32_t* bm = reinterpret_cast<uint32_t*>(smem);
    uint32_t* wpre = bm + kBmWords;
    uint32_t* vc = wpre + kBmWords;
    uint2* seg = reinterpret_cast<uint2*>(vc + kPart);
    const uint32_t b = job.x, s = job.y, n = job.z;
    const bool part = job.w != kUnset;
    if (b >= p.num_buckets || n > kPart || s > p.item_cap || n > p.item_cap - s ||
        (part && job.w >= p.huge_cap)) {
        if (t == 0) set_status(p.hdr, MMBEV_DEV_BOUNDS);
        return;   // uniform over the block
    }
    const uint2* it = p.items + s;
    const bool in_regs = n <= kBT * kIl;   // else the passes read the items again
    const uint32_t nwords = (1u << p.bucket_log2) >= 32u ? (1u << p.bucket_log2) >> 5 : 1u;
    const int lane = t & 31;
    const uint32_t lt = (1u << lane) - 1u;
    // Items are read in rounds of kBT * kIl (the loop bounds are uniform over
    // the block, so whole warps run every collective). Lanes of a warp that
    // meet the same shared-memory word combine their update first.
    uint2 e[kIl];
#pragma unroll
    for (uint32_t c = 0; c < kIl; ++c) {
        const uint32_t i = t + c * kBT;
        e[c] = i < n ? it[i] : make_uint2(kUnset, kUnset);
    }
    // 1. the job's occupancy bitmap
    for (uint32_t w = t; w < nwords; w += kBT) bm[w] = 0u;
    __syncthreads();
    for (uint32_t r0 = 0; r0 < n; r0 += kBT * kIl) {
        if (r0 != 0u) {
#pragma unroll
            for (uint32_t c = 0; c < kIl; ++c) {
                const uint32_t i = r0 + c * kBT + t;
                e[c] = i < n ? it[i] : make_uint2(kUnset, kUnset);
            }
        }
#pragma unroll
        for (uint32_t c = 0; c < kIl; ++c) {
            const uint32_t lo = e[c].x != kUnset ? item_lo(p, e[c].y) : kUnset;
            const uint32_t grp = __match_any_sync(kFull, lo);
            if (lo != kUnset && lane == __ffs(grp) - 1) atomicOr(&bm[lo >> 5], 1u << (lo & 31));
        }
    }
    __syncthreads();
    // 2. word prefixes of its popcounts (two words a thread): voxel v = rank
    // of the low bits
    uint32_t nv = 0;
    {
        uint32_t pc = 0;
        for (uint32_t w = (uint32_t)t * 2; w < (uint32_t)t * 2 + 2; ++w)
            if (w < nwords) pc += __popc(bm[w]);
        uint32_t run = block_exclusive_scan(pc, s_warp, &nv);
        for (uint32_t w = (uint32_t)t * 2; w < (uint32_t)t * 2 + 2; ++w)
            if (w < nwords) {
                wpre[w] = run;
                run += __popc(bm[w]);
                // a part adds its voxels to the split bucket's union (read by
                // the merge, after every part has counted itself done)
                if (part && bm[w]) atomicOr(&p.hbits[(size_t)job.w * kUnionWords + w], bm[w]);
            }
    }
    for (uint32_t v = t; v < nv; v += kBT) vc[v] = 0u;
    __syncthreads();
    // 3. points per voxel
    for (uint32_t r0 = 0; r0 < n; r0 += kBT * kIl) {
        if (!in_regs) {
#pragma unroll
            for (uint32_t c = 0; c < kIl; ++c) {
                const uint32_t i = r0 + c * kBT + t;
                e[c] = i < n ? it[i] : make_uint2(kUnset, kUnset);
            }
        }
#pragma unroll
        for (uint32_t c = 0; c < kIl; ++c) {
            const uint32_t v = e[c].x != kUnset ? voxel_of(bm, wpre, item_lo(p, e[c].y)) : kUnset;
            const uint32_t grp = __match_any_sync(kFull, v);
            if (v != kUnset && lane == __ffs(grp) - 1) atomicAdd(&vc[v], (uint32_t)__popc(grp));
        }
    }
    __syncthreads();
    // 4. their exclusive prefix, in place (a contiguous run of voxels a thread)
    {
        const uint32_t per = (nv + kBT - 1) / kBT;
        const uint32_t v0 = (uint32_t)t * per;
        uint32_t sum = 0;
        for (uint32_t k = 0; k < per; ++k)
            if (v0 + k < nv) sum += vc[v0 + k];
        uint32_t tot = 0;
        uint32_t run = block_exclusive_scan(sum, s_warp, &tot);
        for (uint32_t k = 0; k < per; ++k)
            if (v0 + k < nv) {
                const uint32_t x = vc[v0 + k];
                vc[v0 + k] = run;
                run += x;
            }
    }
    __syncthreads();
    // 5. every point into its voxel's run; afterwards vc[v] is the run's end
    for (uint32_t r0 = 0; r0 < n; r0 += kBT * kIl) {
        if (!in_regs) {
#pragma unroll
            for (uint32_t c = 0; c < kIl; ++c) {
                const uint32_t i = r0 + c * kBT + t;
                e[c] = i < n ? it[i] : make_uint2(kUnset, kUnset);
            }
        }
#pragma unroll
        for (uint32_t c = 0; c < kIl; ++c) {
            const uint32_t v = e[c].x != kUnset ? voxel_of(bm, wpre, item_lo(p, e[c].y)) : kUnset;
            const uint32_t grp = __match_any_sync(kFull, v);
            const int leader = __ffs(grp) - 1;
            uint32_t base = 0;
            if (v != kUnset && lane == leader) base = atomicAdd(&vc[v], (uint32_t)__popc(grp));
            base = __shfl_sync(kFull, base, leader);
            const uint32_t at = base + __popc(grp & lt);
            if (v != kUnset && at < n) seg[at] = e[c];
        }
    }
    __syncthreads();
    // 6. voxels of at most 32 points a thread each, then those of up to
    // 1,024 a warp each, then larger ones the whole block each. A whole
    // bucket's go to vdesc and vitems; a part's to the part lists (pdesc, and
    // the .x words of its own items, all read by now).
    __shared__ uint32_t s_huge[kHugeList + 1];   // voxels of more than kWarpMax points
    __shared__ uint32_t s_dense[kDenseList + 1];  // voxels of 33 .. kWarpMax points
    if (t == 0) {
        s_huge[kHugeList] = 0u;
        s_dense[kDenseList] = 0u;
    }
    __syncthreads();
    uint4* desc = (part ? p.pdesc : p.vdesc) + s;
    auto kept_out = [&](uint32_t st) -> KeptOut {
        if (part) return KeptOut{reinterpret_cast<uint32_t*>(p.items + s + st), 2u, s + st};
        return KeptOut{p.vitems + s + st, 1u, s + st};
    };
    for (uint32_t v = t; v < nv; v += kBT) {
        const uint32_t st = v ? vc[v - 1] : 0u, cnt = vc[v] - st;
        if (cnt > kWarpMax) {
            const uint32_t k = atomicAdd(&s_huge[kHugeList], 1u);
            if (k < kHugeList) s_huge[k] = v;
        } else if (cnt > 32u) {
            const uint32_t k = atomicAdd(&s_dense[kDenseList], 1u);
            if (k < kDenseList) s_dense[k] = v;
        }
    }
    for (uint32_t i = t; i < n; i += kBT) select_small(p, seg, i, bm, wpre, vc, kept_out, desc);
    __syncthreads();
    const uint32_t nh = s_huge[kHugeList];
    const uint32_t nd = min(s_dense[kDenseList], kDenseList);   // never more: see kDenseList
    for (uint32_t k = warp; k < nd; k += kBT / 32) {
        const uint32_t v = s_dense[k];
        const uint32_t st = v ? vc[v - 1] : 0u, cnt = vc[v] - st;
        select_by_warp<BH>(p, seg, st, cnt, kept_out(st), desc + v);
    }
    if (nh > kHugeList)   // huge voxels beyond the list's room, by warps
        for (uint32_t v = warp; v < nv; v += kBT / 32) {
            const uint32_t st = v ? vc[v - 1] : 0u, cnt = vc[v] - st;
            if (cnt > kWarpMax) select_by_warp<BH>(p, seg, st, cnt, kept_out(st), desc + v);
        }
    if (nh <= kHugeList) {
        for (uint32_t k = 0; k < nh; ++k) {   // block-uniform
            const uint32_t v = s_huge[k];
            const uint32_t st = v ? vc[v - 1] : 0u, cnt = vc[v] - st;
            select_by_block<BH>(p, seg, st, cnt, kept_out(st), desc + v, bm);   // bm, wpre: free now
        }
    }
    __syncthreads();
    if (!part) {
        if (t == 0) publish_bucket(p, b, nv);
        return;
    }
    // a part: its voxel count (the merge stage combines the parts)
    if (t == 0) p.pnv[jidx] = nv;
}

// A bucket of at most 32 points by one warp, in registers: lane i holds
// point i. A point's rank in its voxel (by position) is the number of the
// voxel's points with a smaller position; the voxel's first point (rank 0)
// stands for it, so the voxel's index is the number of first points with a
// smaller lin, and its kept positions start after the kept positions of
// those voxels. A point of rank < K writes its own position there.
__device__ void bucket_tiny(const Params& p, const uint4& job) {
    const int lane = threadIdx.x & 31;
    const uint32_t b = job.x, s = job.y, n = job.z;
    if (b >= p.num_buckets || n > 32u || s > p.item_cap || n > p.item_cap - s) {
        if (lane == 0) set_status(p.hdr, MMBEV_DEV_BOUNDS);
        return;
    }
    const bool act = (uint32_t)lane < n;
    const uint2 e = act ? p.items[s + lane] : make_uint2(kUnset, kUnset);
    const uint32_t lo = act ? item_lo(p, e.y) : kUnset;
    const uint32_t rk = e.y >> 16;
    const uint32_t grp = __match_any_sync(kFull, lo);
    const uint32_t K = (uint32_t)p.K;
    uint32_t r = 0, mr = kUnset;
    for (uint32_t j = 0; j < n; ++j) {   // warp-uniform
        const uint32_t pj = __shfl_sync(kFull, e.x, j);
        const uint32_t rj = __shfl_sync(kFull, rk, j);
        if ((grp >> j) & 1u) {
            r += pj < e.x;
            mr = min(mr, rj);
        }
    }
    const uint32_t cnt = __popc(grp);
    const uint32_t kept = min(cnt, K);
    const uint32_t firsts = __ballot_sync(kFull, act && r == 0u);
    uint32_t v = 0, koff = 0;
    for (uint32_t m = firsts; m; m &= m - 1u) {   // warp-uniform
        const int l = __ffs(m) - 1;
        const uint32_t ol = __shfl_sync(kFull, lo, l);
        const uint32_t ok = __shfl_sync(kFull, kept, l);
        if (ol < lo) {
            ++v;
            koff += ok;
        }
    }
    if (act && r < K) p.vitems[s + koff + r] = e.x;
    if (act && r == 0u) p.vdesc[s + v] = make_uint4(s + koff, cnt, lo, mr);
    if (lane == 0) publish_bucket(p, b, __popc(firsts));
    __syncwarp();
}

// A warp job (at most kWarpJobMax points): one bucket by one warp, in its
// own piece of shared memory; a lane keeps up to eight of its items in
// registers. job = {bucket, first item, points, -}.
template <int BH>
__device__ void bucket_by_warp(const Params& p, const uint4& job, unsigned char* piece) {
    constexpr uint32_t kPer = kWarpJobMax / 32;   // 8
    const int lane = threadIdx.x & 31;
    const uint32_t lt = (1u << lane) - 1u;
    uint32_t* bm = reinterpret_cast<uint32_t*>(piece);
    uint32_t* wpre = bm + kBmWords;
    uint32_t* vc = wpre + kBmWords;
    uint2* seg = reinterpret_cast<uint2*>(vc + kWarpJobMax);
    const uint32_t b = job.x, s = job.y, n = job.z;
    if (b >= p.num_buckets || n > kWarpJobMax || s > p.item_cap || n > p.item_cap - s) {
        if (lane == 0) set_status(p.hdr, MMBEV_DEV_BOUNDS);
        return;
    }
    const uint32_t nwords = (1u << p.bucket_log2) >= 32u ? (1u << p.bucket_log2) >> 5 : 1u;
    const uint32_t wpl = (nwords + 31) / 32;   // words a lane
    uint2 e[kPer];
#pragma unroll
    for (uint32_t c = 0; c < kPer; ++c) {
        const uint32_t i = (uint32_t)lane + 32u * c;
        e[c] = i < n ? p.items[s + i] : make_uint2(kUnset, kUnset);
    }
    for (uint32_t w = lane; w < nwords; w += 32) bm[w] = 0u;
    __syncwarp();
#pragma unroll
    for (uint32_t c = 0; c < kPer; ++c)
        if (e[c].x != kUnset) atomicOr(&bm[item_lo(p, e[c].y) >> 5], 1u << (e[c].y & 31));
    __syncwarp();
    uint32_t pc = 0;
    for (uint32_t k = 0; k < wpl; ++k) {
        const uint32_t w = (uint32_t)lane * wpl + k;
        if (w < nwords) pc += __popc(bm[w]);
    }
    uint32_t nv = 0;
    uint32_t run = warp_exclusive_scan(pc, &nv);
    for (uint32_t k = 0; k < wpl; ++k) {
        const uint32_t w = (uint32_t)lane * wpl + k;
        if (w < nwords) {
            wpre[w] = run;
            run += __popc(bm[w]);
        }
    }
#pragma unroll
    for (uint32_t c = 0; c < kPer; ++c) vc[lane + 32 * c] = 0u;
    __syncwarp();
    uint32_t v[kPer];
#pragma unroll
    for (uint32_t c = 0; c < kPer; ++c) {
        v[c] = e[c].x != kUnset ? voxel_of(bm, wpre, item_lo(p, e[c].y)) : kUnset;
        const uint32_t grp = __match_any_sync(kFull, v[c]);
        if (v[c] != kUnset && lane == __ffs(grp) - 1) atomicAdd(&vc[v[c]], (uint32_t)__popc(grp));
    }
    __syncwarp();
    {   // exclusive prefix of vc[0..nv) in place, a run of kPer a lane
        uint32_t x[kPer], sum = 0;
#pragma unroll
        for (uint32_t c = 0; c < kPer; ++c) {
            x[c] = vc[lane * kPer + c];
            sum += x[c];
        }
        uint32_t tot = 0;
        uint32_t r = warp_exclusive_scan(sum, &tot);
        __syncwarp();
#pragma unroll
        for (uint32_t c = 0; c < kPer; ++c) {
            vc[lane * kPer + c] = r;
            r += x[c];
        }
    }
    __syncwarp();
#pragma unroll
    for (uint32_t c = 0; c < kPer; ++c) {
        const uint32_t grp = __match_any_sync(kFull, v[c]);
        const int leader = __ffs(grp) - 1;
        uint32_t base = 0;
        if (v[c] != kUnset && lane == leader) base = atomicAdd(&vc[v[c]], (uint32_t)__popc(grp));
        base = __shfl_sync(kFull, base, leader);
        if (v[c] != kUnset) seg[base + __popc(grp & lt)] = e[c];
    }
    __syncwarp();
    uint4* desc = p.vdesc + s;
    auto kept_out = [&](uint32_t st) { return KeptOut{p.vitems + s + st, 1u, s + st}; };
    for (uint32_t i = lane; i < n; i += 32) select_small(p, seg, i, bm, wpre, vc, kept_out, desc);
    for (uint32_t v0 = 0; v0 < nv; v0 += 32) {   // warp-uniform: voxels of more than 32 points
        bool dense = false;
        if (v0 + (uint32_t)lane < nv) {
            const uint32_t vv = v0 + (uint32_t)lane;
            dense = vc[vv] - (vv ? vc[vv - 1] : 0u) > 32u;
        }
        for (uint32_t m = __ballot_sync(kFull, dense); m; m &= m - 1u) {
            const uint32_t vv = v0 + (uint32_t)(__ffs(m) - 1);
            const uint32_t st = vv ? vc[vv - 1] : 0u, cnt = vc[vv] - st;
            select_by_warp<BH>(p, seg, st, cnt, KeptOut{p.vitems + s + st, 1u, s + st}, desc + vv);
        }
    }
    if (lane == 0) publish_bucket(p, b, nv);
    __syncwarp();
}

// Every block first takes block jobs, one at a time from a counter; thread
// 0 fetches the next job's descriptor and the ticket of the one after while
// the current job is worked on, so no thread waits on them. Then each warp
// takes warp jobs from a second counter the same way, so that warps whose
// block was busy longest take the fewest.
template <int BH>
__global__ void __launch_bounds__(kBT, (BH <= 12 ? 8 : 2)) k_buckets(Params p) {
    extern __shared__ __align__(16) unsigned char smem[];
    __shared__ uint32_t s_warp[kBT / 32];
    __shared__ uint4 s_job;
    __shared__ uint32_t s_jidx;
    pdl_wait();
    const int t = threadIdx.x, warp = t >> 5;
    // tickets: the parts first (so that the merges of the split buckets can
    // start early), then the block jobs, largest class first (the longest
    // jobs do not come last)
    const uint32_t np = min(p.hdr->n_parts, p.part_cap);
    uint32_t nl[3];
#pragma unroll
    for (int q = 0; q < 3; ++q) nl[q] = min(p.hdr->n_large[q], p.job_cap);
    const uint32_t ns = min(p.hdr->n_small, p.num_buckets);
    const uint4 none = make_uint4(kUnset, 0u, 0u, 0u);
    auto job_at = [&](uint32_t k) -> uint4 {
        if (k < np) return p.hjobs[k];
        k -= np;
#pragma unroll
        for (int q = 0; q < 3; ++q) {
            if (k < nl[q]) return p.jobs[(size_t)q * p.job_cap + k];
            k -= nl[q];
        }
        return none;
    };
    uint4 d = none;
    uint32_t jcur = 0, jnext = 0;
    if (t == 0) {
        jcur = atomicAdd(&p.hdr->large_ticket, 1u);
        d = job_at(jcur);
        jnext = atomicAdd(&p.hdr->large_ticket, 1u);
    }
    for (;;) {
        if (t == 0) {
            s_job = d;
            s_jidx = jcur;
        }
        __syncthreads();
        const uint4 job = s_job;
        const uint32_t jidx = s_jidx;
        __syncthreads();   // every thread has its job before s_job is written again
        if (job.x == kUnset) break;
        if (t == 0) {
            d = job_at(jnext);
            jcur = jnext;
            jnext = atomicAdd(&p.hdr->large_ticket, 1u);
        }
        bucket_by_block<BH>(p, job, jidx, smem, s_warp);
    }
    // Then the warp jobs, by ticket: the next job's descriptor and the ticket
    // after it are requested before the current job and used after it.
    unsigned char* piece = smem + (size_t)warp * kWarpSmem;
    const int lane = t & 31;
    uint32_t k = 0, kn = 0;
    if (lane == 0) {
        k = atomicAdd(&p.hdr->small_ticket, 1u);
        kn = atomicAdd(&p.hdr->small_ticket, 1u);
    }
    k = __shfl_sync(kFull, k, 0);
    kn = __shfl_sync(kFull, kn, 0);
    uint4 sj = k < ns ? p.sjobs[k] : none;
    while (k < ns) {   // warp-uniform
        const uint4 next = kn < ns ? p.sjobs[kn] : none;
        uint32_t knn = 0;
        if (lane == 0 && kn < ns) knn = atomicAdd(&p.hdr->small_ticket, 1u);
        if (sj.z <= 32u) bucket_tiny(p, sj);
        else bucket_by_warp<BH>(p, sj, piece);
        sj = next;
        k = kn;
        kn = k < ns ? __shfl_sync(kFull, knn, 0) : ns;
    }
}

// ------------------------------------------------------------------ stage 5

// Merge blocks: one split bucket at a time, with most of the SM's shared
// memory. The union of the parts' voxels (each part ORed its own into hbits)
// gives the bucket's voxels. A pass over the parts' entries adds up each
// voxel's count, takes its minimum rank and counts its candidates (each
// part's K smallest positions of it); a scan places every voxel's
// candidates, a second pass gathers them there, and each voxel's K smallest
// positions are selected from its own candidates (a thread for up to 32, a
// warp beyond). When the candidates of all voxels exceed the buffer they are
// gathered for a window of voxels at a time; a single voxel with more
// candidates than the buffer holds inserts them into K slots (kmin_insert).
// A large split bucket is merged by several blocks, each a range of its
// bitmap words (of its low lin bits): each counts all the bucket's voxels,
// for the kept offsets, and gathers and selects only its own.
constexpr uint32_t kMergeGroup = 1024;            // parts whose entry prefix is held at once
constexpr size_t kMergeSmem = 200 * 1024;         // dynamic shared memory of a merge block
constexpr uint32_t kStash = 2048;                 // entries a task keeps for its gather

template <int B>
__host__ __device__ constexpr int merge_threads() { return B <= 12 ? 1024 : B <= 32 ? 512 : 256; }

template <int B>
__global__ void __launch_bounds__(merge_threads<B>(), 1) k_merge(Params p) {
    constexpr int MT = merge_threads<B>();
    constexpr int TB = B < 32 ? B : 32;            // a thread's voxels have at most 32 candidates
    extern __shared__ __align__(16) uint32_t msm[];
    __shared__ uint32_t s_warp[MT / 32];
    __shared__ uint32_t s_ppre[kMergeGroup + 1];
    __shared__ uint32_t s_x, s_nst;
    pdl_wait();
    const int t = threadIdx.x, lane = t & 31, warp = t >> 5;
    const uint32_t nh = min(p.hdr->n_huge, p.huge_cap);
    const uint32_t K = (uint32_t)p.K;
    const uint32_t nwords = (1u << p.bucket_log2) >= 32u ? (1u << p.bucket_log2) >> 5 : 1u;
    const uint32_t lomask = (1u << p.bucket_log2) - 1u;
    uint32_t* bm = msm;
    uint32_t* wpre = bm + kBmWords;
    uint32_t* vcount = wpre + kBmWords;
    const uint32_t nt = min(p.hdr->n_mtasks, p.mtask_cap);
    for (uint32_t f = blockIdx.x; f < nt; f += gridDim.x) {   // block-uniform
        // task: range tw of TW (of the bitmap words) of split bucket h
        const uint2 task = p.mtasks[f];
        const uint32_t h = task.x, tw = task.y & 0xFFFFu, TW = task.y >> 16;
        if (h >= nh || tw >= TW || TW > nwords) {
            if (t == 0) set_status(p.hdr, MMBEV_DEV_BOUNDS);
            continue;
        }
        const uint32_t j0 = p.hj0[h];
        const uint32_t b = j0 < p.part_cap ? p.hjobs[j0].x : kUnset;
        if (b >= p.num_buckets) {
            if (t == 0) set_status(p.hdr, MMBEV_DEV_BOUNDS);
            continue;
        }
        const uint32_t s = p.boff[b], n = p.bcnt[b];
        const uint32_t P = (n + kPart - 1) / kPart;
        if (j0 + P > p.part_cap || s > p.item_cap || n > p.item_cap - s) {
            if (t == 0) set_status(p.hdr, MMBEV_DEV_BOUNDS);
            continue;
        }
        // 1. the union bitmap and its word prefixes
        uint32_t pc = 0;
        if ((uint32_t)t < nwords) {
            bm[t] = __ldcg(p.hbits + (size_t)h * kUnionWords + t);
            pc = __popc(bm[t]);
        }
        uint32_t nv = 0;
        const uint32_t wex = block_exclusive_scan(pc, s_warp, &nv);
        if ((uint32_t)t < nwords) wpre[t] = wex;
        uint32_t* vmr = vcount + nv;     // minimum rank
        uint32_t* vcc = vmr + nv;        // candidates, then their offsets, then cursors
        uint32_t* kof = vcc + nv;        // kept offsets
        const uint32_t sto = (2u * kBmWords + 4u * nv + 3u) & ~3u;   // the stash, 16-byte aligned
        uint4* stash = reinterpret_cast<uint4*>(msm + sto);          // the task's own entries
        uint32_t* cand = msm + sto + 4u * kStash;
        uint32_t cap = (uint32_t)(kMergeSmem / 4) - sto - 4u * kStash;
        uint32_t stash_cap = kStash;
        if (p.merge_limit) {   // test hook: a smaller buffer and stash
            cap = max(K, min(cap, p.merge_limit));
            stash_cap = min(kStash, p.merge_limit / 4u);
        }
        if (t == 0) s_nst = 0u;
        for (uint32_t v = t; v < nv; v += MT) {
            vcount[v] = 0u;
            vmr[v] = kUnset;
            vcc[v] = 0u;
        }
        __syncthreads();
        // the task's voxels: those of its words
        const uint32_t wa = tw * nwords / TW, wb = (tw + 1) * nwords / TW;
        const uint32_t v_lo = wpre[wa], v_hi = wb < nwords ? wpre[wb] : nv;
        // s_ppre[k] = entries of parts g0 .. g0+k-1; returns their total
        auto group_prefix = [&](uint32_t g0, uint32_t g1) -> uint32_t {
            const uint32_t ng = g1 - g0;
            uint32_t carry = 0;
            for (uint32_t c0 = 0; c0 < ng; c0 += MT) {   // block-uniform
                const uint32_t q = g0 + c0 + t;
                const uint32_t nq =
                    c0 + t < ng ? min(__ldcg(p.pnv + j0 + q), min(kPart, n - q * kPart)) : 0u;
                uint32_t tot = 0;
                const uint32_t e = block_exclusive_scan(nq, s_warp, &tot);
                if (c0 + t < ng) s_ppre[c0 + t] = carry + e;
                carry += tot;
            }
            if (t == 0) s_ppre[ng] = carry;
            __syncthreads();
            return carry;
        };
        // every entry {first kept position, count, lo, minimum rank} of the
        // parts, two a thread in flight: f(entry, its voxel)
        auto for_entries = [&](auto&& f) {
            for (uint32_t g0 = 0; g0 < P; g0 += kMergeGroup) {   // block-uniform
                const uint32_t g1 = min(P, g0 + kMergeGroup), ng = g1 - g0;
                const uint32_t ne = group_prefix(g0, g1);
                constexpr int U = 4;
                for (uint32_t i0 = t; i0 < ne; i0 += MT * U) {
                    uint4 d[U];
#pragma unroll
                    for (int u = 0; u < U; ++u) {
                        const uint32_t i = i0 + (uint32_t)u * MT;
                        d[u] = make_uint4(0u, 0u, 0u, kUnset);
                        if (i < ne) {
                            uint32_t a = 0, z = ng;   // s_ppre[a] <= i < s_ppre[a + 1]
                            while (z - a > 1) {
                                const uint32_t mid = (a + z) >> 1;
                                if (s_ppre[mid] <= i) a = mid; else z = mid;
                            }
                            d[u] = __ldcg(p.pdesc + s + (size_t)(g0 + a) * kPart + (i - s_ppre[a]));
                        }
                    }
#pragma unroll
                    for (int u = 0; u < U; ++u)
                        if (d[u].y != 0u) f(d[u], voxel_of(bm, wpre, d[u].z & lomask));
                }
                __syncthreads();   // s_ppre of the next group
            }
        };
        // the kept positions of entry d (its candidates, in any order), eight
        // loads in flight: g(j, position); stops early when g returns false
        auto for_candidates = [&](const uint4& d, auto&& g) {
            const uint32_t kq = min(d.y, K);
            if (d.x > p.item_cap || kq > p.item_cap - d.x) {
                set_status(p.hdr, MMBEV_DEV_BOUNDS);
                return;
            }
            const uint32_t* kp = reinterpret_cast<const uint32_t*>(p.items + d.x);   // .x words
            for (uint32_t q0 = 0; q0 < kq; q0 += 8) {
                uint32_t c[8];
#pragma unroll
                for (int k = 0; k < 8; ++k) c[k] = q0 + k < kq ? __ldcg(kp + 2 * (q0 + k)) : kUnset;
                bool go = true;
#pragma unroll
                for (int k = 0; k < 8; ++k)
                    if (go && q0 + k < kq) go = g(q0 + k, c[k]);
                if (!go) break;
            }
        };
        // 2. counts, minimum ranks, candidates per voxel; the task's own
        // entries kept aside for the gather (up to kStash of them)
        for_entries([&](const uint4& d, uint32_t v) {
            atomicAdd(&vcount[v], d.y);
            atomicMin(&vmr[v], d.w);
            atomicAdd(&vcc[v], min(d.y, K));
            if (v >= v_lo && v < v_hi) {
                const uint32_t k = atomicAdd(&s_nst, 1u);
                if (k < stash_cap) stash[k] = d;
            }
        });
        const uint32_t nst = s_nst;
        // the task's entries: from the stash when they all fit, else read again
        auto for_task_entries = [&](auto&& f) {
            if (nst <= stash_cap) {
                for (uint32_t i = t; i < nst; i += MT) {
                    const uint4 d = stash[i];
                    f(d, voxel_of(bm, wpre, d.z & lomask));
                }
                __syncthreads();
            } else {
                for_entries(f);
            }
        };
        // 3. candidate offsets into vcc, kept offsets into kof (runs of
        // consecutive voxels a thread)
        uint32_t C = 0;
        {
            const uint32_t per = (nv + MT - 1) / MT;
            const uint32_t v0 = (uint32_t)t * per;
            uint32_t cs = 0, ks = 0;
            for (uint32_t k = 0; k < per; ++k)
                if (v0 + k < nv) {
                    cs += vcc[v0 + k];
                    ks += min(vcount[v0 + k], K);
                }
            uint32_t kt = 0;
            uint32_t ce = block_exclusive_scan(cs, s_warp, &C);
            uint32_t ke = block_exclusive_scan(ks, s_warp, &kt);
            for (uint32_t k = 0; k < per; ++k)
                if (v0 + k < nv) {
                    const uint32_t x = vcc[v0 + k];
                    vcc[v0 + k] = ce;
                    ce += x;
                    kof[v0 + k] = ke;
                    ke += min(vcount[v0 + k], K);
                }
        }
        __syncthreads();
        // voxel v's descriptor; its kept positions go to vitems[s + kof[v] ..]
        auto put_desc = [&](uint32_t v) {
            p.vdesc[s + v] = make_uint4(s + kof[v], vcount[v], lo_of_voxel(bm, wpre, nwords, v), vmr[v]);
        };
        // 4. windows of the task's voxels whose candidates fit the buffer
        uint32_t w0 = v_lo;
        while (w0 < v_hi) {   // block-uniform
            if (t == 0) {
                const uint32_t base = vcc[w0];
                uint32_t a = w0, z = v_hi + 1;   // largest a with coff(a) - base <= cap
                while (z - a > 1) {
                    const uint32_t mid = (a + z) >> 1;
                    if ((mid < nv ? vcc[mid] : C) - base <= cap) a = mid; else z = mid;
                }
                s_x = a;
            }
            __syncthreads();
            uint32_t w1 = s_x;
            const uint32_t base = vcc[w0];
            const uint32_t next = w0 + 1 < nv ? vcc[w0 + 1] : C;
            __syncthreads();   // every thread has read vcc[w0] before the gather moves it
            if (w1 == w0) {
                // one voxel with more candidates than the buffer: K slots
                for (uint32_t j = t; j < K; j += MT) cand[j] = kUnset;
                __syncthreads();
                for_task_entries([&](const uint4& d, uint32_t v) {
                    if (v != w0) return;
                    for_candidates(d, [&](uint32_t, uint32_t c) {
                        kmin_insert(cand, K, c);
                        return true;
                    });
                });
                const uint32_t kept = min(vcount[w0], K);
                if (kof[w0] + kept <= n) {
                    for (uint32_t j = t; j < kept; j += MT) p.vitems[s + kof[w0] + j] = cand[j];
                } else if (t == 0) {
                    set_status(p.hdr, MMBEV_DEV_BOUNDS);
                }
                if (t == 0) {
                    put_desc(w0);
                    vcc[w0] = next;   // as if gathered
                }
                w1 = w0 + 1;
            } else {
                for_task_entries([&](const uint4& d, uint32_t v) {
                    if (v < w0 || v >= w1) return;
                    const uint32_t at = atomicAdd(&vcc[v], min(d.y, K)) - base;
                    for_candidates(d, [&](uint32_t j, uint32_t c) {
                        cand[at + j] = c;
                        return true;
                    });
                });
                // voxel v's candidates: cand[st, en)
                auto range = [&](uint32_t v, uint32_t& st, uint32_t& en) {
                    st = v == w0 ? 0u : vcc[v - 1] - base;
                    en = vcc[v] - base;
                };
                for (uint32_t v = w0 + t; v < w1; v += MT) {
                    uint32_t st, en;
                    range(v, st, en);
                    if (en - st > 32u) continue;
                    uint32_t best[TB];
#pragma unroll
                    for (int j = 0; j < TB; ++j) best[j] = kUnset;
                    for (uint32_t i = st; i < en; ++i) sorted_insert<TB>(best, cand[i]);
                    const uint32_t kept = kof[v] + min(vcount[v], K) <= n ? min(vcount[v], K) : 0u;
                    if (kept < min(vcount[v], K)) set_status(p.hdr, MMBEV_DEV_BOUNDS);
#pragma unroll
                    for (int j = 0; j < TB; ++j)
                        if ((uint32_t)j < kept) p.vitems[s + kof[v] + j] = best[j];
                    put_desc(v);
                }
                for (uint32_t v = w0 + warp; v < w1; v += MT / 32) {   // warp-uniform
                    uint32_t st, en;
                    range(v, st, en);
                    if (en - st <= 32u) continue;
                    uint32_t best[B];
#pragma unroll
                    for (int j = 0; j < B; ++j) best[j] = kUnset;
                    for (uint32_t i = st + lane; i < en; i += 32) sorted_insert<B>(best, cand[i]);
                    const uint32_t kept = kof[v] + min(vcount[v], K) <= n ? min(vcount[v], K) : 0u;
                    if (lane == 0 && kept < min(vcount[v], K)) set_status(p.hdr, MMBEV_DEV_BOUNDS);
                    for (uint32_t j = 0; j < kept; ++j) {
                        const uint32_t m = __reduce_min_sync(kFull, best[0]);
                        if (best[0] == m) {   // positions are distinct: one lane owns m
                            p.vitems[s + kof[v] + j] = m;
#pragma unroll
                            for (int c = 0; c + 1 < B; ++c) best[c] = best[c + 1];
                            best[B - 1] = kUnset;
                        }
                    }
                    if (lane == 0) put_desc(v);
                }
            }
            __syncthreads();
            w0 = w1;
        }
        if (t == 0 && tw == 0) publish_bucket(p, b, nv);
        __syncthreads();
    }
}

template <int B>
cudaError_t launch_merge_t(const Params& p, int num_sms, bool pdl, cudaStream_t st) {
    static std::atomic<int> configured[64];
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    if (dev < 0 || dev >= 64 || !configured[dev].load(std::memory_order_acquire)) {
        e = cudaFuncSetAttribute(k_merge<B>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                 (int)kMergeSmem);
        if (e != cudaSuccess) return e;
        if (dev >= 0 && dev < 64) configured[dev].store(1, std::memory_order_release);
    }
    return launch_k(k_merge<B>, dim3(num_sms), dim3(merge_threads<B>()), kMergeSmem, st, pdl, p);
}

// ------------------------------------------------------------------ stage 6

constexpr int kOutThreads = 256;
constexpr uint32_t kOutSlice = 1u << kSliceLog2;   // buckets a block
static_assert(kOutSlice == 2 * kOutThreads, "two buckets a thread");

// record: {x', y', z', intensity} {dt, rank, -, -}
__device__ __forceinline__ void add_record(float (&acc)[5], const uint4& a, float dt) {
    acc[0] = __fadd_rn(acc[0], __uint_as_float(a.x));
    acc[1] = __fadd_rn(acc[1], __uint_as_float(a.y));
    acc[2] = __fadd_rn(acc[2], __uint_as_float(a.z));
    acc[3] = __fadd_rn(acc[3], __uint_as_float(a.w));
    acc[4] = __fadd_rn(acc[4], dt);
}

// Features of the record at position q (clamped into the array; a position
// outside it is reported).
__device__ __forceinline__ void load_record(const Params& p, uint32_t q, uint4& a, float& dt) {
    if (q >= p.rec_cap) set_status(p.hdr, MMBEV_DEV_BOUNDS);
    const uint4* rec = p.records + 2 * (size_t)min(q, p.rec_cap - 1u);
    a = __ldg(rec);
    dt = __ldg(reinterpret_cast<const float*>(rec + 1));
}

// Voxel d of bucket-in-frame bi into output row `row` of frame f: the mean
// of its kept points' records (their positions ascend in vitems), summed in
// that order in fp32 and divided once, its count and its coordinates.
template <int B>
__device__ __forceinline__ void finalize_voxel(const Params& p, uint32_t f, uint32_t row,
                                               uint32_t bi, const uint4& d) {
    const uint32_t kept = min(d.y, (uint32_t)p.K);
    if (d.x > p.item_cap || kept > p.item_cap - d.x) {
        set_status(p.hdr, MMBEV_DEV_BOUNDS);
        return;
    }
    uint32_t pos[B];
#pragma unroll
    for (int j = 0; j < B; ++j) pos[j] = (uint32_t)j < kept ? p.vitems[d.x + j] : kUnset;
    sort_small<B>(pos);   // kept positions come in any order; the sum goes by index
    constexpr int R = B < 2 ? B : 2;   // record loads in flight (more warps beat more loads a warp)
    float acc[5] = {0.f, 0.f, 0.f, 0.f, 0.f};
#pragma unroll
    for (int j0 = 0; j0 < B; j0 += R) {
        if ((uint32_t)j0 >= kept) break;
        uint4 ra[R];
        float dt[R];
#pragma unroll
        for (int c = 0; c < R; ++c)
            if ((uint32_t)(j0 + c) < kept) load_record(p, pos[j0 + c], ra[c], dt[c]);
#pragma unroll
        for (int c = 0; c < R; ++c)
            if ((uint32_t)(j0 + c) < kept) add_record(acc, ra[c], dt[c]);
    }
    const size_t r = (size_t)f * (uint32_t)p.max_voxels + row;
    const float fc = (float)kept;
#pragma unroll
    for (int c = 0; c < 5; ++c) p.out_feats[r * 5 + c] = __fdiv_rn(acc[c], fc);
    const uint32_t lin = (bi << p.bucket_log2) | d.z;
    const uint32_t q = udiv(p.div_nx, lin);      // cz * ny + cy
    const uint32_t cz = udiv(p.div_ny, q);
    p.out_coords[r * 3 + 0] = (int32_t)cz;
    p.out_coords[r * 3 + 1] = (int32_t)(q - cz * p.dims[1]);
    p.out_coords[r * 3 + 2] = (int32_t)(lin - q * p.dims[0]);
    p.out_counts[r] = (int32_t)kept;
}

// The non-empty buckets among [c0, c0 + kOutSlice) of frame f (two a
// thread) go to s_list as {bucket in frame, exclusive voxel prefix within
// the range + carry, voxels, first item}; returns how many, and the range's
// voxel total in *tot. Every thread must call it.
__device__ __forceinline__ uint32_t list_range(const Params& p, uint32_t b0, uint32_t c0,
                                               uint32_t hi, uint32_t carry, uint4* s_list,
                                               uint32_t* s_warp, uint32_t* tot) {
    const int t = threadIdx.x;
    const uint32_t bi0 = c0 + 2u * (uint32_t)t, bi1 = bi0 + 1u;
    const uint32_t u0 = bi0 < hi ? p.ucnt[b0 + bi0] : 0u;
    const uint32_t u1 = bi1 < hi ? p.ucnt[b0 + bi1] : 0u;
    const uint32_t s0 = u0 ? p.boff[b0 + bi0] : 0u;
    const uint32_t s1 = u1 ? p.boff[b0 + bi1] : 0u;
    const uint32_t e = block_exclusive_scan(u0 + u1, s_warp, tot);
    const uint32_t ne = (uint32_t)(u0 != 0u) + (uint32_t)(u1 != 0u);
    uint32_t nne = 0;
    uint32_t at = block_exclusive_scan(ne, s_warp, &nne);
    if (u0) s_list[at++] = make_uint4(bi0, carry + e, u0, s0);
    if (u1) s_list[at] = make_uint4(bi1, carry + e + u0, u1, s1);
    __syncthreads();
    return nne;
}

// A frame over the cap, by one block: histogram of the voxels' minimum ranks,
// threshold rank r* and quota q, then every kept voxel's row in ascending lin.
template <int B>
__device__ void capped_frame(const Params& p, uint32_t f, uint32_t* s_hist, uint32_t* s_warp,
                             uint4* s_list) {
    const int t = threadIdx.x, lane = t & 31, warp = t >> 5;
    constexpr int nwarps = kOutThreads / 32;
    const uint32_t Bf = p.buckets_per_frame;
    const uint32_t b0 = f * Bf;
    const uint32_t rn = (uint32_t)(p.frame_roi_off[f + 1] - p.frame_roi_off[f]);   // background rank
    const uint32_t maxv = (uint32_t)p.max_voxels;
    __shared__ uint32_t s_rstar, s_q;
    for (uint32_t r = t; r <= rn; r += kOutThreads) s_hist[r] = 0u;
    __syncthreads();
    uint32_t tot = 0;
    for (uint32_t c0 = 0; c0 < Bf; c0 += kOutSlice) {
        const uint32_t nne = list_range(p, b0, c0, Bf, 0u, s_list, s_warp, &tot);
        for (uint32_t k = warp; k < nne; k += nwarps) {
            const uint4 L = s_list[k];
            for (uint32_t v = lane; v < L.z; v += 32)
                atomicAdd(&s_hist[min(p.vdesc[L.w + v].w, rn)], 1u);
        }
        __syncthreads();
    }
    if (t == 0) {
        uint32_t cum = 0, rstar = rn, q = 0;
        for (uint32_t r = 0; r <= rn; ++r) {
            if (cum + s_hist[r] >= maxv) {
                rstar = r;
                q = maxv - cum;
                break;
            }
            cum += s_hist[r];
        }
        s_rstar = rstar;
        s_q = q;
    }
    __syncthreads();
    const uint32_t rstar = s_rstar, q = s_q;
    // voxels below r* and at r* per non-empty bucket
    for (uint32_t c0 = 0; c0 < Bf; c0 += kOutSlice) {
        const uint32_t nne = list_range(p, b0, c0, Bf, 0u, s_list, s_warp, &tot);
        for (uint32_t k = warp; k < nne; k += nwarps) {
            const uint4 L = s_list[k];
            uint32_t below = 0, tie = 0;
            for (uint32_t v = lane; v < L.z; v += 32) {
                const uint32_t r = min(p.vdesc[L.w + v].w, rn);
                below += r < rstar;
                tie += r == rstar;
            }
#pragma unroll
            for (int o = 16; o > 0; o >>= 1) {
                below += __shfl_xor_sync(kFull, below, o);
                tie += __shfl_xor_sync(kFull, tie, o);
            }
            if (lane == 0) p.bcap[b0 + L.x] = make_uint2(below, tie);
        }
        __syncthreads();
    }
    // rows in ascending lin: a voxel below r* takes (below-voxels before it)
    // + min(ties before it, q); a tie voxel is kept when fewer than q ties
    // precede it
    uint32_t carry_a = 0, carry_c = 0;
    for (uint32_t c0 = 0; c0 < Bf; c0 += kOutSlice) {
        const uint32_t bi0 = c0 + 2u * (uint32_t)t, bi1 = bi0 + 1u;
        const uint2 x0 = bi0 < Bf && p.ucnt[b0 + bi0] ? p.bcap[b0 + bi0] : make_uint2(0u, 0u);
        const uint2 x1 = bi1 < Bf && p.ucnt[b0 + bi1] ? p.bcap[b0 + bi1] : make_uint2(0u, 0u);
        uint32_t ta = 0, tc = 0;
        const uint32_t ea = block_exclusive_scan(x0.x + x1.x, s_warp, &ta);
        const uint32_t ec = block_exclusive_scan(x0.y + x1.y, s_warp, &tc);
        if (bi0 < Bf) p.bcap[b0 + bi0] = make_uint2(carry_a + ea, carry_c + ec);
        if (bi1 < Bf) p.bcap[b0 + bi1] = make_uint2(carry_a + ea + x0.x, carry_c + ec + x0.y);
        carry_a += ta;
        carry_c += tc;
        __syncthreads();
        const uint32_t nne = list_range(p, b0, c0, Bf, 0u, s_list, s_warp, &tot);
        for (uint32_t k = warp; k < nne; k += nwarps) {
            const uint4 L = s_list[k];
            const uint2 pre = p.bcap[b0 + L.x];
            uint32_t a = pre.x, c = pre.y;
            for (uint32_t v0 = 0; v0 < L.z; v0 += 32) {
                const uint32_t v = v0 + lane;
                uint4 d = make_uint4(0u, 0u, 0u, kUnset);
                uint32_t r = kUnset;
                if (v < L.z) {
                    d = p.vdesc[L.w + v];
                    r = min(d.w, rn);
                }
                const uint32_t lt = (1u << lane) - 1u;
                const uint32_t mb = __ballot_sync(kFull, v < L.z && r < rstar);
                const uint32_t mt = __ballot_sync(kFull, v < L.z && r == rstar);
                const uint32_t ab = a + __popc(mb & lt), cb = c + __popc(mt & lt);
                if (v < L.z) {
                    uint32_t row = kUnset;
                    if (r < rstar) row = ab + min(cb, q);
                    else if (r == rstar && cb < q) row = ab + cb;
                    if (row != kUnset) {
                        if (row < maxv) finalize_voxel<B>(p, f, row, L.x, d);
                        else set_status(p.hdr, MMBEV_DEV_BOUNDS);
                    }
                }
                a += __popc(mb);
                c += __popc(mt);
            }
        }
        __syncthreads();
    }
    if (t == 0) p.out_nvox[f] = (int32_t)maxv;
}

// Rows a chunk of the output stage: one a thread.
constexpr uint32_t kChunkRows = kOutThreads;
constexpr uint32_t kMaxSlices = (1u << (32 - kBucketLog2Max)) >> kSliceLog2;   // 1,024

// Persistent blocks. Each first takes frames over the cap (a block each),
// then chunks of kChunkRows output rows of the other frames, so that every
// block gets about the same number of voxels however they crowd into a few
// buckets. A chunk locates its rows' buckets from the frame's slice sums and
// a scan of the bucket counts of the slices it touches; then each thread
// finalizes one row.
template <int B>
__global__ void __launch_bounds__(kOutThreads, (B <= 12 ? 6 : 2)) k_output(Params p) {
    __shared__ uint32_t s_warp[kOutThreads / 32];
    __shared__ uint32_t s_cpre[kMaxFrames + 1];   // chunks before each frame
    __shared__ uint32_t s_spre[kMaxSlices + 1];   // voxels before each slice of a frame
    __shared__ uint32_t s_hist[kMaxRoisPerFrame + 2];
    __shared__ uint4 s_list[kOutSlice];
    pdl_wait();
    const int t = threadIdx.x;
    const uint32_t F = (uint32_t)p.num_frames;
    const uint32_t S = p.out_slices;
    const uint32_t Bf = p.buckets_per_frame;
    const uint32_t maxv = (uint32_t)p.max_voxels;
    // chunks per frame (none for a frame over the cap), and their prefix
    {
        uint32_t u[4], c[4], sum = 0;
#pragma unroll
        for (int k = 0; k < 4; ++k) {
            const uint32_t f = 4u * (uint32_t)t + k;
            u[k] = f < F ? p.ftot[f] : 0u;
            c[k] = u[k] <= maxv ? (u[k] + kChunkRows - 1) / kChunkRows : 0u;
            sum += c[k];
            if (blockIdx.x == 0 && f < F) p.out_nvox[f] = (int32_t)min(u[k], maxv);
        }
        uint32_t tot = 0;
        uint32_t run = block_exclusive_scan(sum, s_warp, &tot);
#pragma unroll
        for (int k = 0; k < 4; ++k) {
            const uint32_t f = 4u * (uint32_t)t + k;
            if (f < F) s_cpre[f] = run;
            run += c[k];
        }
        if (t == 0) s_cpre[F] = tot;
        __syncthreads();
    }
    const uint32_t C = s_cpre[F];
    for (uint32_t f = blockIdx.x; f < F; f += gridDim.x)   // block-uniform
        if (p.ftot[f] > maxv) capped_frame<B>(p, f, s_hist, s_warp, s_list);
    for (uint32_t c = blockIdx.x; c < C; c += gridDim.x) {
        uint32_t lo = 0, hi = F;   // s_cpre[lo] <= c < s_cpre[hi]
        while (hi - lo > 1) {
            const uint32_t mid = (lo + hi) >> 1;
            if (s_cpre[mid] <= c) lo = mid; else hi = mid;
        }
        const uint32_t f = lo;
        const uint32_t U = p.ftot[f];
        const uint32_t r0 = (c - s_cpre[f]) * kChunkRows, r1 = min(U, r0 + kChunkRows);
        // voxels before each slice of the frame
        {
            uint32_t x[4], sum = 0;
#pragma unroll
            for (int k = 0; k < 4; ++k) {
                const uint32_t j = 4u * (uint32_t)t + k;
                x[k] = j < S ? p.ssum[f * S + j] : 0u;
                sum += x[k];
            }
            uint32_t tot = 0;
            uint32_t run = block_exclusive_scan(sum, s_warp, &tot);
#pragma unroll
            for (int k = 0; k < 4; ++k) {
                const uint32_t j = 4u * (uint32_t)t + k;
                if (j < S) s_spre[j] = run;
                run += x[k];
            }
            if (t == 0) s_spre[S] = tot;
            __syncthreads();
        }
        uint32_t j0 = 0, jh = S;   // the slice holding row r0: s_spre[j0] <= r0 < s_spre[j0 + 1]
        while (jh - j0 > 1) {
            const uint32_t mid = (j0 + jh) >> 1;
            if (s_spre[mid] <= r0) j0 = mid; else jh = mid;
        }
        for (uint32_t j = j0; j < S && s_spre[j] < r1; ++j) {   // block-uniform
            const uint32_t b0 = f * Bf, cb = j * kOutSlice;
            uint32_t tot = 0;
            const uint32_t nne = list_range(p, b0, cb, min(Bf, cb + kOutSlice), s_spre[j], s_list,
                                            s_warp, &tot);
            // this thread's row, if it lies in the slice
            const uint32_t row = r0 + (uint32_t)t;
            if (row < r1 && row >= s_spre[j] && row < s_spre[j + 1] && nne > 0) {
                uint32_t a = 0, z = nne;   // s_list[a].y <= row < s_list[a + 1].y
                while (z - a > 1) {
                    const uint32_t mid = (a + z) >> 1;
                    if (s_list[mid].y <= row) a = mid; else z = mid;
                }
                const uint4 L = s_list[a];   // bucket in frame, first row, voxels, first item
                const uint32_t v = row - L.y;
                if (v < L.z && row < maxv && L.w + v < p.item_cap)
                    finalize_voxel<B>(p, f, row, L.x, p.vdesc[L.w + v]);
                else
                    set_status(p.hdr, MMBEV_DEV_BOUNDS);
            }
            __syncthreads();   // s_list is rebuilt for the next slice
        }
    }
}

}  // namespace

cudaError_t launch_bucket_scan(const Params& p, bool pdl, cudaStream_t st) {
    if (p.scan_tiles == 0) return cudaSuccess;
    return launch_k(k_bucket_scan, dim3(p.scan_tiles), dim3(kScanThreads), 0, st, pdl, p);
}

cudaError_t launch_bucket_scatter(const Params& p, int num_sms, bool pdl, cudaStream_t st) {
    return launch_k(k_bucket_scatter, dim3(num_sms * 8), dim3(kThreads), 0, st, pdl, p);
}

template <int BH>
cudaError_t launch_buckets_t(const Params& p, int num_sms, bool pdl, cudaStream_t st) {
    static std::atomic<int> configured[64];
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    if (dev < 0 || dev >= 64 || !configured[dev].load(std::memory_order_acquire)) {
        e = cudaFuncSetAttribute(k_buckets<BH>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                 (int)kBlockSmem);
        if (e != cudaSuccess) return e;
        if (dev >= 0 && dev < 64) configured[dev].store(1, std::memory_order_release);
    }
    const int per_sm = BH <= 12 ? 8 : 2;
    return launch_k(k_buckets<BH>, dim3(num_sms * per_sm), dim3(kBT), kBlockSmem, st, pdl, p);
}

cudaError_t launch_buckets(const Params& p, int num_sms, bool pdl, cudaStream_t st) {
    if (p.K <= 4) return launch_buckets_t<4>(p, num_sms, pdl, st);
    if (p.K <= 12) return launch_buckets_t<12>(p, num_sms, pdl, st);
    if (p.K <= 32) return launch_buckets_t<32>(p, num_sms, pdl, st);
    return launch_buckets_t<kMaxK>(p, num_sms, pdl, st);
}

cudaError_t launch_merge(const Params& p, int num_sms, bool pdl, cudaStream_t st) {
    if (p.K <= 4) return launch_merge_t<4>(p, num_sms, pdl, st);
    if (p.K <= 12) return launch_merge_t<12>(p, num_sms, pdl, st);
    if (p.K <= 32) return launch_merge_t<32>(p, num_sms, pdl, st);
    return launch_merge_t<kMaxK>(p, num_sms, pdl, st);
}

cudaError_t launch_output(const Params& p, int num_sms, bool pdl, cudaStream_t st) {
    const dim3 grid(num_sms * (p.K <= 12 ? 6 : 2)), block(kOutThreads);
    if (p.K <= 4) return launch_k(k_output<4>, grid, block, 0, st, pdl, p);
    if (p.K <= 12) return launch_k(k_output<12>, grid, block, 0, st, pdl, p);
    if (p.K <= 32) return launch_k(k_output<32>, grid, block, 0, st, pdl, p);
    return launch_k(k_output<kMaxK>, grid, block, 0, st, pdl, p);
}

uint32_t output_slices(uint32_t buckets_per_frame) {
    return (buckets_per_frame + kOutSlice - 1) / kOutSlice;
}

}  // namespace mmbev
