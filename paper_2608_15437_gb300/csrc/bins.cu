// Stages 2-5: voxel dedup (S3), cap and canonical order (S4), first-K mean
// features (S5) of the path (Alg. 1 "Voxelize" and "VoxelFeatureEncoder";
// Sec. IV-F hard voxelization; Sec. IV-C mandatory ROIs first).
//
// The classify pass has counted every kept point into its bucket (2^LB
// consecutive linear indices of one frame; bucket b = frame * Bf + lin >> LB,
// so buckets ascend with (frame, lin)) and numbered its arrival there. Then:
//
//   scan     (stage 2)  exclusive prefix of the bucket counts over the whole
//                       call (one pass, tiles of 4,096 buckets chained by
//                       decoupled look-back: a tile publishes its total, then
//                       its inclusive prefix once its predecessors' are
//                       known), and the non-empty buckets listed as small
//                       (at most 64 points) or large.
//   scatter  (stage 3)  a counting sort of the kept points by bucket: entry
//                       {position, low lin bits | rank} goes to item
//                       boff[bucket] + arrival. No atomics.
//   buckets  (stage 4)  each bucket alone: its voxels are the distinct low
//                       lin bits of its points, ranked by a shared-memory
//                       occupancy bitmap (popcount prefix), so voxel v of the
//                       bucket is the v-th smallest lin; a counting sort by
//                       voxel gives each voxel's points; the voxel keeps its
//                       K smallest record positions (= smallest point
//                       indices), sums their features in that order in fp32
//                       and divides once. Results go to temps[boff + v] in
//                       ascending lin, the voxel count to ucnt[bucket]. A
//                       warp takes a small bucket, a block a large one (its
//                       point lists in shared memory up to 2,048 points, else
//                       in global scratch).
//   output   (stage 5)  per frame: the voxel counts of its buckets, scanned,
//                       give every voxel its output row (ascending lin). A
//                       frame over max_voxels keeps the max_voxels smallest
//                       by (minimum rank, lin): a histogram of minimum ranks
//                       gives the threshold rank r* and the quota q of
//                       rank-r* voxels that fit; rank-r* voxels are kept in
//                       ascending lin until q are taken.
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

__device__ __forceinline__ void write_temp(VoxTemp* t, const float (&acc)[5], uint32_t cnt,
                                           uint32_t minrank, uint32_t lo) {
    const float fc = (float)cnt;
    float4* d = reinterpret_cast<float4*>(t);
    d[0] = make_float4(__fdiv_rn(acc[0], fc), __fdiv_rn(acc[1], fc), __fdiv_rn(acc[2], fc),
                       __fdiv_rn(acc[3], fc));
    d[1] = make_float4(__fdiv_rn(acc[4], fc), __uint_as_float(cnt), __uint_as_float(minrank),
                       __uint_as_float(lo));
}

// Voxel of low lin bits `lo` in a bucket: its rank among the bucket's
// distinct low bits, from the occupancy bitmap and its word prefixes.
__device__ __forceinline__ uint32_t voxel_of(const uint32_t* bm, const uint32_t* wpre, uint32_t lo) {
    const uint32_t w = lo >> 5;
    return wpre[w] + __popc(bm[w] & ((1u << (lo & 31)) - 1u));
}

// One voxel by one thread: entries seg[start, start+cnt) {position, lo |
// rank << 16} (any order, cnt <= B or the B smallest kept). Keeps the K
// smallest positions in order, sums their records, writes the temp.
template <int B>
__device__ __forceinline__ void voxel_by_thread(const Params& p, const uint2* seg, uint32_t start,
                                                uint32_t cnt, VoxTemp* out) {
    uint32_t best[B];
#pragma unroll
    for (int j = 0; j < B; ++j) best[j] = kUnset;
    uint32_t mr = kUnset, lo = 0;
    for (uint32_t i = 0; i < cnt; ++i) {
        const uint2 e = seg[start + i];
        sorted_insert<B>(best, e.x);
        mr = min(mr, e.y >> 16);
        lo = e.y & 0xFFFFu;
    }
    const uint32_t kept = min(cnt, (uint32_t)p.K);
    constexpr int R = B < 3 ? B : 3;   // record loads in flight
    float acc[5] = {0.f, 0.f, 0.f, 0.f, 0.f};
#pragma unroll
    for (int j0 = 0; j0 < B; j0 += R) {
        if ((uint32_t)j0 >= kept) break;
        uint4 ra[R];
        float dt[R];
#pragma unroll
        for (int c = 0; c < R; ++c)
            if ((uint32_t)(j0 + c) < kept) load_record(p, best[j0 + c], ra[c], dt[c]);
#pragma unroll
        for (int c = 0; c < R; ++c)
            if ((uint32_t)(j0 + c) < kept) add_record(acc, ra[c], dt[c]);
    }
    write_temp(out, acc, kept, mr, lo);
}

// One voxel by a whole warp (any count): each lane keeps the B smallest
// positions of every 32nd entry, K rounds of a warp minimum pick the K
// smallest in ascending order (the j-th goes to lane j % 32, register
// j / 32), the lanes load those records together and every lane adds them
// up in order; lane 0 writes.
template <int B>
__device__ __forceinline__ void voxel_by_warp(const Params& p, const uint2* seg, uint32_t start,
                                              uint32_t cnt, VoxTemp* out) {
    const int lane = threadIdx.x & 31;
    uint32_t best[B];
#pragma unroll
    for (int j = 0; j < B; ++j) best[j] = kUnset;
    uint32_t mr = kUnset;
    for (uint32_t i = lane; i < cnt; i += 32) {
        const uint2 e = seg[start + i];
        sorted_insert<B>(best, e.x);
        mr = min(mr, e.y >> 16);
    }
    mr = __reduce_min_sync(kFull, mr);
    const uint32_t lo = seg[start].y & 0xFFFFu;
    const int kept = (int)min(cnt, (uint32_t)p.K);
    uint32_t mine[2] = {kUnset, kUnset};
    for (int j = 0; j < kept; ++j) {
        const uint32_t m = __reduce_min_sync(kFull, best[0]);
        if (lane == (j & 31)) mine[j >> 5] = m;
        if (best[0] == m) {   // positions are distinct: one lane owns m
#pragma unroll
            for (int c = 0; c + 1 < B; ++c) best[c] = best[c + 1];
            best[B - 1] = kUnset;
        }
    }
    float acc[5] = {0.f, 0.f, 0.f, 0.f, 0.f};
    for (int half = 0; half * 32 < kept; ++half) {
        uint4 ra = make_uint4(0u, 0u, 0u, 0u);
        float rdt = 0.f;
        if (half * 32 + lane < kept) load_record(p, mine[half], ra, rdt);
        const int m = kept - half * 32 < 32 ? kept - half * 32 : 32;
        for (int j = 0; j < m; ++j) {
            uint4 a;
            a.x = __shfl_sync(kFull, ra.x, j);
            a.y = __shfl_sync(kFull, ra.y, j);
            a.z = __shfl_sync(kFull, ra.z, j);
            a.w = __shfl_sync(kFull, ra.w, j);
            add_record(acc, a, __shfl_sync(kFull, rdt, j));
        }
    }
    if (lane == 0) write_temp(out, acc, (uint32_t)kept, mr, lo);
}

// ------------------------------------------------------------------ stage 2

constexpr int kScanThreads = 1024;
static_assert(kScanTile == kScanThreads * 4, "four buckets a thread");
constexpr unsigned long long kAggFlag = 1ull << 32;    // tile total published
constexpr unsigned long long kIncFlag = 2ull << 32;    // tile inclusive prefix published

// Append the buckets of `take` (one lane each) to list `dst` of length
// counter `cnt` with one atomic per warp.
__device__ __forceinline__ void warp_append(bool take, uint32_t b, uint32_t* cnt, uint32_t* dst,
                                            uint32_t cap, Header* hdr) {
    const int lane = threadIdx.x & 31;
    const uint32_t m = __ballot_sync(kFull, take);
    if (!m) return;
    const int leader = __ffs(m) - 1;
    uint32_t base = 0;
    if (lane == leader) base = atomicAdd(cnt, (uint32_t)__popc(m));
    base = __shfl_sync(kFull, base, leader);
    if (take) {
        const uint32_t at = base + __popc(m & ((1u << lane) - 1u));
        if (at < cap) dst[at] = b;
        else set_status(hdr, MMBEV_DEV_BOUNDS);
    }
}

__global__ void __launch_bounds__(kScanThreads) k_bucket_scan(Params p) {
    __shared__ uint32_t s_warp[kScanThreads / 32];
    __shared__ uint32_t s_tile, s_base;
    pdl_wait();
    const int t = threadIdx.x;
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
    if (t == 0) {
        unsigned long long* st = p.scan_state;
        uint32_t base = 0;
        if (tile == 0) {
            atomicExch(&st[0], kIncFlag | total);
        } else {
            atomicExch(&st[tile], kAggFlag | total);
            // look back: add the predecessors' totals until one has
            // published its inclusive prefix (bounded waits)
            int64_t j = (int64_t)tile - 1;
            while (j >= 0) {
                unsigned long long w = 0ull;
                uint32_t spins = 0;
                while (((w = ld_acquire(&st[j])) >> 32) == 0ull) {
                    if (++spins >= kSpinLimit) break;
                }
                if ((w >> 32) == 0ull) {   // gave up: the results are void
                    set_status(p.hdr, MMBEV_DEV_WAIT_TIMEOUT);
                    break;
                }
                base += (uint32_t)w;
                if ((w & kIncFlag) != 0ull) break;
                --j;
            }
            atomicExch(&st[tile], kIncFlag | (unsigned long long)(base + total));
        }
        s_base = base;
    }
    __syncthreads();
    uint32_t run = s_base + excl;
#pragma unroll
    for (int k = 0; k < 4; ++k) {
        const uint32_t b = b0 + k;
        if (b < B) {
            p.boff[b] = run;
            p.ucnt[b] = 0u;
            if (b == B - 1u) p.boff[B] = run + c[k];
        }
        run += c[k];
        warp_append(b < B && c[k] > kSmallMax, b, &p.hdr->n_large, p.large, B, p.hdr);
        warp_append(b < B && c[k] > 0u && c[k] <= kSmallMax, b, &p.hdr->n_small, p.small, B,
                    p.hdr);
    }
}

// ------------------------------------------------------------------ stage 3

constexpr int kThreads = 256;

// Prefix sums of the classify blocks' list lengths (off[0..G]) and the
// first plist entry of each list (list l starts at tile t_begin(l) * 2048).
struct Lists {
    uint32_t off[kMaxClsGrid + 1];
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
    uint32_t total = 0;
    uint32_t run = block_exclusive_scan(sum, s_warp, &total);
#pragma unroll
    for (int k = 0; k < 4; ++k) {
        const uint32_t l = (uint32_t)threadIdx.x * 4 + k;
        if (l <= G) L.off[l] = run;
        run += c[k];
    }
    __syncthreads();
    return L.off[G];
}

// plist index of the i-th entry of the concatenated lists.
__device__ __forceinline__ size_t list_entry(const Params& p, const Lists& L, uint32_t i) {
    uint32_t lo = 0, hi = p.cls_grid;  // L.off[lo] <= i < L.off[hi]
    while (hi - lo > 1) {
        const uint32_t mid = (lo + hi) >> 1;
        if (L.off[mid] <= i) lo = mid; else hi = mid;
    }
    return (size_t)L.start[lo] + (i - L.off[lo]);
}

__global__ void __launch_bounds__(kThreads) k_bucket_scatter(Params p) {
    __shared__ Lists L;
    __shared__ uint32_t s_warp[kThreads / 32];
    pdl_wait();
    const uint32_t M = lists_scan(p, L, s_warp);
    const uint32_t gs = gridDim.x * blockDim.x;
    constexpr int U = 4;   // entries a thread has in flight
    for (uint32_t i0 = blockIdx.x * blockDim.x + threadIdx.x; i0 < M; i0 += U * gs) {
        uint4 e[U];
#pragma unroll
        for (int u = 0; u < U; ++u) {
            const uint32_t i = i0 + (uint32_t)u * gs;
            e[u] = i < M ? __ldcs(p.plist + list_entry(p, L, i)) : make_uint4(kUnset, 0u, 0u, 0u);
        }
        uint32_t at[U];
#pragma unroll
        for (int u = 0; u < U; ++u)
            at[u] = e[u].x < p.num_buckets ? __ldg(p.boff + e[u].x) + e[u].w : kUnset;
#pragma unroll
        for (int u = 0; u < U; ++u) {
            if (e[u].x == kUnset) continue;
            if (at[u] < p.item_cap) p.items[at[u]] = make_uint2(e[u].y, e[u].z);
            else set_status(p.hdr, MMBEV_DEV_BOUNDS);
        }
    }
}

// ------------------------------------------------------------------ stage 4

// Shared memory of a block on a large bucket (the warps on small buckets
// carve the same bytes into per-warp pieces).
constexpr int kBmWords = (1 << kBucketLog2Max) / 32;    // 256
constexpr uint32_t kMaxVox = 1u << kBucketLog2Max;      // voxels a bucket can hold
constexpr size_t kLargeSmem = (size_t)kBmWords * 4 * 2 + (size_t)kMaxVox * 4 +
                              (size_t)kSegSmem * sizeof(uint2);
constexpr size_t kWarpSmem = (size_t)kBmWords * 4 * 2 + kSmallMax * 4 + kSmallMax * sizeof(uint2);
static_assert(kWarpSmem * (kThreads / 32) <= kLargeSmem, "the small-bucket pieces fit");

// A large bucket by the whole block.
template <int BL, int BH>
__device__ void bucket_by_block(const Params& p, uint32_t b, unsigned char* smem, uint32_t* s_warp) {
    const int t = threadIdx.x, lane = t & 31, warp = t >> 5;
    uint32_t* bm = reinterpret_cast<uint32_t*>(smem);
    uint32_t* wpre = bm + kBmWords;
    uint32_t* vc = wpre + kBmWords;
    uint2* seg_s = reinterpret_cast<uint2*>(vc + kMaxVox);
    const uint32_t s = p.boff[b];
    const uint32_t n = p.bcnt[b];
    if (s > p.item_cap || n > p.item_cap - s) {
        if (t == 0) set_status(p.hdr, MMBEV_DEV_BOUNDS);
        return;   // uniform over the block
    }
    const uint2* it = p.items + s;
    uint2* seg = n <= kSegSmem ? seg_s : p.seg2 + s;
    const uint32_t nwords = (1u << p.bucket_log2) >= 32u ? (1u << p.bucket_log2) >> 5 : 1u;
    // 1. the bucket's occupancy bitmap
    for (uint32_t w = t; w < nwords; w += kThreads) bm[w] = 0u;
    __syncthreads();
    for (uint32_t i = t; i < n; i += kThreads) {
        const uint32_t lo = it[i].y & 0xFFFFu;
        atomicOr(&bm[lo >> 5], 1u << (lo & 31));
    }
    __syncthreads();
    // 2. word prefixes of its popcounts: voxel v = rank of the low bits
    uint32_t nv = 0;
    const uint32_t pc = (uint32_t)t < nwords ? __popc(bm[t]) : 0u;
    const uint32_t wp = block_exclusive_scan(pc, s_warp, &nv);
    if ((uint32_t)t < nwords) wpre[t] = wp;
    for (uint32_t v = t; v < nv; v += kThreads) vc[v] = 0u;
    __syncthreads();
    // 3. points per voxel
    for (uint32_t i = t; i < n; i += kThreads)
        atomicAdd(&vc[voxel_of(bm, wpre, it[i].y & 0xFFFFu)], 1u);
    __syncthreads();
    // 4. their exclusive prefix, in place (a contiguous run of voxels a thread)
    {
        const uint32_t per = (nv + kThreads - 1) / kThreads;
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
    for (uint32_t i = t; i < n; i += kThreads) {
        const uint2 e = it[i];
        const uint32_t at = atomicAdd(&vc[voxel_of(bm, wpre, e.y & 0xFFFFu)], 1u);
        if (at < n) seg[at] = e;
    }
    __syncthreads();
    // 6. voxels of at most 32 points a thread each, then the others a warp each
    VoxTemp* out = p.temps + s;
    for (uint32_t v = t; v < nv; v += kThreads) {
        const uint32_t st = v ? vc[v - 1] : 0u, cnt = vc[v] - st;
        if (cnt <= 32) voxel_by_thread<BL>(p, seg, st, cnt, out + v);
    }
    for (uint32_t v = warp; v < nv; v += kThreads / 32) {
        const uint32_t st = v ? vc[v - 1] : 0u, cnt = vc[v] - st;
        if (cnt > 32) voxel_by_warp<BH>(p, seg, st, cnt, out + v);
    }
    if (t == 0) p.ucnt[b] = nv;
    (void)lane;
    __syncthreads();
}

// A small bucket (at most kSmallMax points) by one warp, in its own piece of
// shared memory.
template <int BL, int BH>
__device__ void bucket_by_warp(const Params& p, uint32_t b, unsigned char* piece) {
    const int lane = threadIdx.x & 31;
    uint32_t* bm = reinterpret_cast<uint32_t*>(piece);
    uint32_t* wpre = bm + kBmWords;
    uint32_t* vc = wpre + kBmWords;
    uint2* seg = reinterpret_cast<uint2*>(vc + kSmallMax);
    const uint32_t s = p.boff[b];
    const uint32_t n = min(p.bcnt[b], kSmallMax);
    if (s > p.item_cap || n > p.item_cap - s) {
        if (lane == 0) set_status(p.hdr, MMBEV_DEV_BOUNDS);
        return;
    }
    const uint32_t nwords = (1u << p.bucket_log2) >= 32u ? (1u << p.bucket_log2) >> 5 : 1u;
    const uint32_t wpl = (nwords + 31) / 32;   // words a lane
    const uint2 e0 = (uint32_t)lane < n ? p.items[s + lane] : make_uint2(0u, 0u);
    const uint2 e1 = (uint32_t)lane + 32u < n ? p.items[s + lane + 32] : make_uint2(0u, 0u);
    for (uint32_t w = lane; w < nwords; w += 32) bm[w] = 0u;
    __syncwarp();
    if ((uint32_t)lane < n) atomicOr(&bm[(e0.y & 0xFFFFu) >> 5], 1u << (e0.y & 31));
    if ((uint32_t)lane + 32u < n) atomicOr(&bm[(e1.y & 0xFFFFu) >> 5], 1u << (e1.y & 31));
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
    vc[lane] = 0u;
    vc[lane + 32] = 0u;
    __syncwarp();
    const uint32_t v0 = (uint32_t)lane < n ? voxel_of(bm, wpre, e0.y & 0xFFFFu) : 0u;
    const uint32_t v1 = (uint32_t)lane + 32u < n ? voxel_of(bm, wpre, e1.y & 0xFFFFu) : 0u;
    if ((uint32_t)lane < n) atomicAdd(&vc[v0], 1u);
    if ((uint32_t)lane + 32u < n) atomicAdd(&vc[v1], 1u);
    __syncwarp();
    {   // exclusive prefix of vc[0..64) in place
        const uint32_t a = vc[lane], c = vc[lane + 32];
        uint32_t ta = 0, tc = 0;
        const uint32_t ea = warp_exclusive_scan(a, &ta);
        const uint32_t ec = warp_exclusive_scan(c, &tc);
        __syncwarp();
        vc[lane] = ea;
        vc[lane + 32] = ta + ec;
    }
    __syncwarp();
    if ((uint32_t)lane < n) seg[atomicAdd(&vc[v0], 1u)] = e0;
    if ((uint32_t)lane + 32u < n) seg[atomicAdd(&vc[v1], 1u)] = e1;
    __syncwarp();
    VoxTemp* out = p.temps + s;
    for (uint32_t v = lane; v < nv; v += 32) {
        const uint32_t st = v ? vc[v - 1] : 0u, cnt = vc[v] - st;
        if (cnt <= 32) voxel_by_thread<BL>(p, seg, st, cnt, out + v);
    }
    for (uint32_t v = 0; v < nv; ++v) {   // a bucket of <= 64 points has at most one such voxel
        const uint32_t st = v ? vc[v - 1] : 0u, cnt = vc[v] - st;
        if (cnt > 32) voxel_by_warp<BH>(p, seg, st, cnt, out + v);
    }
    if (lane == 0) p.ucnt[b] = nv;
    __syncwarp();
}

// Every block first takes large buckets, one at a time from a counter, then
// its warps take small ones, one at a time each.
template <int BL, int BH>
__global__ void __launch_bounds__(kThreads, (BH <= 12 ? 4 : 1)) k_buckets(Params p) {
    extern __shared__ __align__(16) unsigned char smem[];
    __shared__ uint32_t s_warp[kThreads / 32];
    __shared__ uint32_t s_job;
    pdl_wait();
    const int t = threadIdx.x, lane = t & 31, warp = t >> 5;
    const uint32_t nl = min(p.hdr->n_large, p.num_buckets);
    const uint32_t ns = min(p.hdr->n_small, p.num_buckets);
    for (;;) {
        if (t == 0) s_job = atomicAdd(&p.hdr->large_ticket, 1u);
        __syncthreads();
        const uint32_t job = s_job;
        __syncthreads();   // every thread has its job before s_job is written again
        if (job >= nl) break;
        bucket_by_block<BL, BH>(p, p.large[job], smem, s_warp);
    }
    unsigned char* piece = smem + (size_t)warp * kWarpSmem;
    for (;;) {
        uint32_t job = 0;
        if (lane == 0) job = atomicAdd(&p.hdr->small_ticket, 1u);
        job = __shfl_sync(kFull, job, 0);
        if (job >= ns) break;
        bucket_by_warp<BL, BH>(p, p.small[job], piece);
    }
}

// ------------------------------------------------------------------ stage 5

constexpr int kOutThreads = 256;
constexpr uint32_t kOutSlice = 2048;   // buckets of a frame per block

// Output row `row` of frame f: voxel temp `tv` of bucket-in-frame bi.
__device__ __forceinline__ void write_row(const Params& p, uint32_t f, uint32_t row, uint32_t bi,
                                          const VoxTemp& tv) {
    const size_t r = (size_t)f * (uint32_t)p.max_voxels + row;
    const uint32_t lin = (bi << p.bucket_log2) | tv.lo;
    const uint32_t q = udiv(p.div_nx, lin);      // cz * ny + cy
    const uint32_t cz = udiv(p.div_ny, q);
#pragma unroll
    for (int c = 0; c < 5; ++c) p.out_feats[r * 5 + c] = tv.f[c];
    p.out_coords[r * 3 + 0] = (int32_t)cz;
    p.out_coords[r * 3 + 1] = (int32_t)(q - cz * p.dims[1]);
    p.out_coords[r * 3 + 2] = (int32_t)(lin - q * p.dims[0]);
    p.out_counts[r] = (int32_t)tv.count;
}

__device__ __forceinline__ VoxTemp load_temp(const VoxTemp* t) {
    const float4* s = reinterpret_cast<const float4*>(t);
    const float4 a = __ldcs(s), c = __ldcs(s + 1);
    VoxTemp v;
    v.f[0] = a.x; v.f[1] = a.y; v.f[2] = a.z; v.f[3] = a.w; v.f[4] = c.x;
    v.count = __float_as_uint(c.y);
    v.minrank = __float_as_uint(c.z);
    v.lo = __float_as_uint(c.w);
    return v;
}

// A frame over the cap, by one block: histogram of the voxels' minimum ranks,
// threshold rank r* and quota q, then every voxel's row in ascending lin.
__device__ void capped_frame(const Params& p, uint32_t f, uint32_t* s_hist, uint32_t* s_warp) {
    const int t = threadIdx.x, lane = t & 31, warp = t >> 5;
    constexpr int nwarps = kOutThreads / 32;
    const uint32_t Bf = p.buckets_per_frame;
    const uint32_t b0 = f * Bf;
    const uint32_t rn = (uint32_t)(p.frame_roi_off[f + 1] - p.frame_roi_off[f]);   // background rank
    const uint32_t maxv = (uint32_t)p.max_voxels;
    __shared__ uint32_t s_rstar, s_q;
    for (uint32_t r = t; r <= rn; r += kOutThreads) s_hist[r] = 0u;
    __syncthreads();
    for (uint32_t bi = warp; bi < Bf; bi += nwarps) {
        const uint32_t b = b0 + bi, nv = p.ucnt[b], s = p.boff[b];
        for (uint32_t v = lane; v < nv; v += 32)
            atomicAdd(&s_hist[min(p.temps[s + v].minrank, rn)], 1u);
    }
    __syncthreads();
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
    // voxels below r* and at r* per bucket
    for (uint32_t bi = warp; bi < Bf; bi += nwarps) {
        const uint32_t b = b0 + bi, nv = p.ucnt[b], s = p.boff[b];
        uint32_t below = 0, tie = 0;
        for (uint32_t v = lane; v < nv; v += 32) {
            const uint32_t r = min(p.temps[s + v].minrank, rn);
            below += r < rstar;
            tie += r == rstar;
        }
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) {
            below += __shfl_xor_sync(kFull, below, o);
            tie += __shfl_xor_sync(kFull, tie, o);
        }
        if (lane == 0) p.bcap[b] = make_uint2(below, tie);
    }
    __syncthreads();
    // their exclusive prefixes over the frame's buckets, in ascending lin
    uint32_t carry_a = 0, carry_c = 0;
    for (uint32_t c0 = 0; c0 < Bf; c0 += kOutThreads) {
        const uint32_t bi = c0 + t;
        const uint2 x = bi < Bf ? p.bcap[b0 + bi] : make_uint2(0u, 0u);
        uint32_t ta = 0, tc = 0;
        const uint32_t ea = block_exclusive_scan(x.x, s_warp, &ta);
        const uint32_t ec = block_exclusive_scan(x.y, s_warp, &tc);
        if (bi < Bf) p.bcap[b0 + bi] = make_uint2(carry_a + ea, carry_c + ec);
        carry_a += ta;
        carry_c += tc;
    }
    __syncthreads();
    // rows: a voxel below r* takes (below-voxels before it) + min(ties before
    // it, q); a tie voxel is kept when fewer than q ties precede it
    for (uint32_t bi = warp; bi < Bf; bi += nwarps) {
        const uint32_t b = b0 + bi, nv = p.ucnt[b], s = p.boff[b];
        if (nv == 0) continue;
        const uint2 pre = p.bcap[b];
        uint32_t a = pre.x, c = pre.y;
        for (uint32_t v0 = 0; v0 < nv; v0 += 32) {
            const uint32_t v = v0 + lane;
            VoxTemp tv;
            uint32_t r = kUnset;
            if (v < nv) {
                tv = load_temp(p.temps + s + v);
                r = min(tv.minrank, rn);
            }
            const uint32_t lt = (1u << lane) - 1u;
            const uint32_t mb = __ballot_sync(kFull, v < nv && r < rstar);
            const uint32_t mt = __ballot_sync(kFull, v < nv && r == rstar);
            const uint32_t ab = a + __popc(mb & lt), cb = c + __popc(mt & lt);
            if (v < nv) {
                if (r < rstar) {
                    const uint32_t row = ab + min(cb, q);
                    if (row < maxv) write_row(p, f, row, bi, tv);
                    else set_status(p.hdr, MMBEV_DEV_BOUNDS);
                } else if (r == rstar && cb < q) {
                    const uint32_t row = ab + cb;
                    if (row < maxv) write_row(p, f, row, bi, tv);
                    else set_status(p.hdr, MMBEV_DEV_BOUNDS);
                }
            }
            a += __popc(mb);
            c += __popc(mt);
        }
    }
    if (t == 0) p.out_nvox[f] = (int32_t)maxv;
}

// Block (f, j) writes the rows of the voxels of the j-th slice of frame f's
// buckets; a frame over the cap is done by its block j = 0 alone.
__global__ void __launch_bounds__(kOutThreads) k_output(Params p, uint32_t slices) {
    __shared__ uint32_t s_warp[kOutThreads / 32];
    __shared__ uint32_t s_hist[kMaxRoisPerFrame + 2];
    __shared__ uint32_t s_pre[kOutThreads];
    pdl_wait();
    const int t = threadIdx.x, lane = t & 31, warp = t >> 5;
    constexpr int nwarps = kOutThreads / 32;
    const uint32_t f = blockIdx.x / slices, j = blockIdx.x % slices;
    const uint32_t Bf = p.buckets_per_frame;
    const uint32_t b0 = f * Bf;
    const uint32_t lo = (uint32_t)((uint64_t)j * Bf / slices);
    const uint32_t hi = (uint32_t)((uint64_t)(j + 1) * Bf / slices);
    // the frame's voxels before the slice and in all
    uint32_t before = 0, all = 0;
    for (uint32_t bi = t; bi < Bf; bi += kOutThreads) {
        const uint32_t u = p.ucnt[b0 + bi];
        all += u;
        if (bi < lo) before += u;
    }
    uint32_t tb = 0, ta = 0;
    (void)block_exclusive_scan(before, s_warp, &tb);
    (void)block_exclusive_scan(all, s_warp, &ta);
    const uint32_t maxv = (uint32_t)p.max_voxels;
    if (ta > maxv) {
        if (j == 0) capped_frame(p, f, s_hist, s_warp);
        return;
    }
    if (j == 0 && t == 0) p.out_nvox[f] = (int32_t)ta;
    // rows of the slice's buckets, kOutThreads buckets at a time
    uint32_t carry = tb;
    for (uint32_t c0 = lo; c0 < hi; c0 += kOutThreads) {
        const uint32_t bi = c0 + t;
        const uint32_t u = bi < hi ? p.ucnt[b0 + bi] : 0u;
        uint32_t tot = 0;
        const uint32_t e = block_exclusive_scan(u, s_warp, &tot);
        s_pre[t] = carry + e;
        __syncthreads();
        const uint32_t nb = min((uint32_t)kOutThreads, hi - c0);
        for (uint32_t k = warp; k < nb; k += nwarps) {
            const uint32_t bb = c0 + k;
            const uint32_t b = b0 + bb, nv = p.ucnt[b], s = p.boff[b], r0 = s_pre[k];
            for (uint32_t v = lane; v < nv; v += 32) {
                const uint32_t row = r0 + v;
                if (row < maxv && s + v < p.item_cap) write_row(p, f, row, bb, load_temp(p.temps + s + v));
                else set_status(p.hdr, MMBEV_DEV_BOUNDS);
            }
        }
        carry += tot;
        __syncthreads();
    }
}

}  // namespace

cudaError_t launch_bucket_scan(const Params& p, bool pdl, cudaStream_t st) {
    if (p.scan_tiles == 0) return cudaSuccess;
    return launch_k(k_bucket_scan, dim3(p.scan_tiles), dim3(kScanThreads), 0, st, pdl, p);
}

cudaError_t launch_bucket_scatter(const Params& p, int num_sms, bool pdl, cudaStream_t st) {
    return launch_k(k_bucket_scatter, dim3(num_sms * 4), dim3(kThreads), 0, st, pdl, p);
}

template <int BL, int BH>
cudaError_t launch_buckets_t(const Params& p, int num_sms, bool pdl, cudaStream_t st) {
    static std::atomic<int> configured[64];
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    if (dev < 0 || dev >= 64 || !configured[dev].load(std::memory_order_acquire)) {
        e = cudaFuncSetAttribute(k_buckets<BL, BH>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                 (int)kLargeSmem);
        if (e != cudaSuccess) return e;
        if (dev >= 0 && dev < 64) configured[dev].store(1, std::memory_order_release);
    }
    const int per_sm = BH <= 12 ? 4 : 1;
    return launch_k(k_buckets<BL, BH>, dim3(num_sms * per_sm), dim3(kThreads), kLargeSmem, st,
                    pdl, p);
}

cudaError_t launch_buckets(const Params& p, int num_sms, bool pdl, cudaStream_t st) {
    if (p.K <= 4) return launch_buckets_t<4, 4>(p, num_sms, pdl, st);
    if (p.K <= 12) return launch_buckets_t<12, 12>(p, num_sms, pdl, st);
    if (p.K <= 32) return launch_buckets_t<32, 32>(p, num_sms, pdl, st);
    return launch_buckets_t<32, kMaxK>(p, num_sms, pdl, st);
}

cudaError_t launch_output(const Params& p, int num_sms, bool pdl, cudaStream_t st) {
    const uint32_t slices = (p.buckets_per_frame + kOutSlice - 1) / kOutSlice;
    (void)num_sms;
    return launch_k(k_output, dim3(p.num_frames * slices), dim3(kOutThreads), 0, st, pdl, p,
                    slices);
}

}  // namespace mmbev
