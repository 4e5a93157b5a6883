// Stage 2: voxel hash insert and dedup (S3 of the path; Alg. 1 "Voxelize"),
// stage 3: the occupied-voxel list, stage 4: per-voxel point lists.
//
// The classify pass leaves, per classify block, a dense list of its kept
// points {lin, frame, record position} (in any order). All three kernels
// here walk the concatenation of those lists; a block finds the list of an
// entry by binary search over the lists' prefix sums in shared memory.
//
// Insert. Persistent blocks; each warp takes 32 consecutive entries at a
// time (the next 32 load while the current ones are inserted), with no
// block barrier in the loop:
//   1. lanes holding the same voxel key are grouped with __match_any_sync
//      (all later warp collectives run on the full warp);
//   2. the group leader finds the key's slot from its home slot (linear
//      probing, at most H probes): a matching key means found, an empty slot
//      is claimed with atomicCAS; it adds the group's size to the slot's
//      point count with one atomicAdd whose old value numbers the group's
//      points (an all-zero slot is empty);
//   3. each lane stores {slot, arrival number} at its entry.
//   A leader that created the slot appends {slot, lin, frame} to its block's
//   sub-list (one shared-memory atomic per warp). No point ever waits on
//   another point's insertion: the voxel's first K points are chosen later,
//   from the complete list.
// Compact. One block per insert block copies that block's sub-list into the
// dense occupied-voxel list at a place taken with one atomicAdd (the list's
// order is immaterial), counts every new voxel into its frame and into its
// ordering bucket (warp-aggregated, recording its position in the bucket),
// and reserves the voxel's segment of `seg` (one atomicAdd per block chunk),
// written into the slot.
// Scatter points. Every entry's record position goes to seg[slot segment +
// arrival number], so each voxel's points end up contiguous. In frames over
// the voxel cap it also lowers the voxel's minimum ROI rank (stored as
// 0xFFFFFFFF - rank) with atomicMax.
#include "mmbev_internal.cuh"

namespace mmbev {
namespace {

constexpr int kThreads = 256;
constexpr int kBlocksPerSm = 8;
// compact: a block takes its insert block's sub-list (about 320 voxels on
// 32 nuScenes-shaped frames) in one pass, so its chain of barriers and
// global atomics runs once
constexpr int kCompactThreads = 512;
constexpr int kFrameWin = 64;
constexpr uint32_t kFull = 0xFFFFFFFFu;

// Prefix sums of the classify blocks' list lengths (off[0..G]) and the
// first plist entry of each list (list l starts at tile t_begin(l) * 2048;
// record positions, and so entries, fit in 32 bits).
struct Lists {
    uint32_t off[kMaxClsGrid + 1];
    uint32_t start[kMaxClsGrid];
};

// Every thread must call it (one barrier). Returns the entry count.
__device__ __forceinline__ uint32_t lists_scan(const Params& p, Lists& L, uint32_t* s_part) {
    const int t = threadIdx.x, lane = t & 31, warp = t >> 5;
    const uint32_t G = p.cls_grid;
    const uint64_t T = (uint64_t)p.num_regions / (kTile / kRegion);
    // kMaxClsGrid <= kThreads * 4: each thread scans up to 4 consecutive lists
    uint32_t c[4], sum = 0;
#pragma unroll
    for (int k = 0; k < 4; ++k) {
        const uint32_t l = (uint32_t)t * 4 + k;
        c[k] = 0;
        if (l < G) {
            const uint64_t t0 = (uint64_t)l * T / G;
            const uint64_t room = ((uint64_t)(l + 1) * T / G - t0) * kTile;
            c[k] = (uint32_t)min((uint64_t)ld_cg(&p.cls_cnt[l]), room);
            L.start[l] = (uint32_t)(t0 * kTile);
        }
        sum += c[k];
    }
    uint32_t v = sum;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        const uint32_t x = __shfl_up_sync(kFull, v, o);
        if (lane >= o) v += x;
    }
    if (lane == 31) s_part[warp] = v;
    __syncthreads();
    uint32_t wbase = 0;
    for (int w = 0; w < warp; ++w) wbase += s_part[w];
    uint32_t run = wbase + v - sum;
#pragma unroll
    for (int k = 0; k < 4; ++k) {
        const uint32_t l = (uint32_t)t * 4 + k;
        if (l <= G) L.off[l] = run;
        run += c[k];
    }
    __syncthreads();
    return L.off[G];
}

// Entry index (into plist / rs) of the i-th entry of the concatenation.
__device__ __forceinline__ size_t list_entry(const Params& p, const Lists& L, uint32_t i) {
    const uint32_t G = p.cls_grid;
    uint32_t lo = 0, hi = G;  // L.off[lo] <= i < L.off[hi]
    while (hi - lo > 1) {
        const uint32_t mid = (lo + hi) >> 1;
        if (L.off[mid] <= i) lo = mid; else hi = mid;
    }
    return (size_t)L.start[lo] + (i - L.off[lo]);
}

__global__ void __launch_bounds__(kThreads, kBlocksPerSm) k_insert(Params p) {
    __shared__ Lists L;
    __shared__ uint32_t s_part[kThreads / 32];
    __shared__ uint32_t s_nnew;
    pdl_wait();
    const int t = threadIdx.x, lane = t & 31;
    if (t == 0) s_nnew = 0;
    const uint32_t M = lists_scan(p, L, s_part);
    // slots in use: a power of two >= 1.25 x the call's kept points
    uint32_t lg = 10;
    if (p.table_log2_fixed > 0) {
        lg = (uint32_t)p.table_log2_fixed;
    } else {
        const uint64_t need = (uint64_t)M * 5 / 4;
        while (lg < p.table_log2 && (1ull << lg) < need) ++lg;
    }
    const uint32_t mask = (uint32_t)((1ull << lg) - 1ull);
    const uint32_t lt = (1u << lane) - 1u;
    uint4* sub = p.newlist + (size_t)blockIdx.x * p.ins_cap;
    const uint32_t nb = (M + 31) / 32;
    const uint32_t gw = (blockIdx.x * kThreads + t) >> 5;
    const uint32_t W = (gridDim.x * kThreads) >> 5;
    // batch g is processed while the warp's next batch loads
    uint32_t g = gw;
    bool act = g * 32 + lane < M;
    size_t e = act ? list_entry(p, L, g * 32 + lane) : 0;
    uint4 a = act ? __ldcs(p.plist + e) : make_uint4(0u, 0u, 0u, 0u);   // lin, frame, pos
    for (; g < nb; g += W) {
        const uint32_t in = (g + W) * 32 + lane;
        const bool actn = g + W < nb && in < M;
        const size_t en = actn ? list_entry(p, L, in) : 0;
        const uint4 an = actn ? __ldcs(p.plist + en) : make_uint4(0u, 0u, 0u, 0u);

        const uint32_t am = __ballot_sync(kFull, act);
        const unsigned long long key = ((unsigned long long)a.y << 32) | a.x;
        uint32_t grp = 1u << lane;
        if (act) grp = __match_any_sync(am, key);
        const int leader = __ffs(grp) - 1;
        bool created = false;
        uint32_t h = kUnset, base = 0;
        if (act && lane == leader) {
            const unsigned long long key1 = key + 1ull;
            h = slot_home(mask, key1);
            bool done = false;
            for (uint32_t probe = 0; probe <= mask; ++probe) {
                const unsigned long long cur = __ldcg(slot_key(p, h));
                if (cur == key1) { done = true; break; }
                if (cur == 0ull) {
                    const unsigned long long old = atomicCAS(slot_key(p, h), 0ull, key1);
                    if (old == 0ull) { created = true; done = true; break; }
                    if (old == key1) { done = true; break; }
                }
                h = (h + 1u) & mask;
            }
            if (!done) {
                set_status(p.hdr, MMBEV_DEV_TABLE_FULL);
                h = kUnset;
            } else {
                base = atomicAdd(slot_cnt(p, h), (uint32_t)__popc(grp));
            }
        }
        h = __shfl_sync(kFull, h, leader);
        base = __shfl_sync(kFull, base, leader);
        if (act) p.rs[e] = make_uint2(h, base + __popc(grp & lt));
        // leaders of new slots append to this block's sub-list
        const uint32_t cm = __ballot_sync(kFull, created);
        if (cm) {
            uint32_t wbase = 0;
            if (lane == __ffs(cm) - 1) wbase = atomicAdd(&s_nnew, (uint32_t)__popc(cm));
            wbase = __shfl_sync(kFull, wbase, __ffs(cm) - 1);
            const uint32_t at = wbase + __popc(cm & lt);
            if (created && at < p.ins_cap) sub[at] = make_uint4(h, a.x, a.y, 0u);
        }
        a = an;
        e = en;
        act = actn;
    }
    __syncthreads();
    if (t == 0) p.blockcount[blockIdx.x] = min(s_nnew, p.ins_cap);
}

__global__ void __launch_bounds__(kCompactThreads) k_compact(Params p) {
    __shared__ uint32_t s_seg[kCompactThreads / 32];
    __shared__ uint32_t s_base, s_segbase;
    __shared__ uint32_t s_fcnt[kFrameWin];
    __shared__ uint32_t s_fmin;
    pdl_wait();
    const int t = threadIdx.x, lane = t & 31, warp = t >> 5;
    const uint32_t b = blockIdx.x;
    const uint4* sub = p.newlist + (size_t)b * p.ins_cap;
    const uint32_t n = min(p.blockcount[b], p.ins_cap);
    if (n == 0) return;
    if (t < kFrameWin) s_fcnt[t] = 0;
    // this block's place in the occupied-voxel list (order is immaterial)
    if (t == 0) {
        s_fmin = sub[0].z;
        s_base = atomicAdd(&p.hdr->num_occ, n);
    }
    __syncthreads();
    const uint32_t base = s_base;
    for (uint32_t i0 = 0; i0 < n; i0 += kCompactThreads) {
        const uint32_t i = i0 + t;
        const bool act = i < n;
        uint4 e = make_uint4(0u, 0u, 0u, 0u);
        uint32_t bk = 0, d = base + i, cnt = 0;
        if (act) {
            e = sub[i];
            bk = e.z * p.buckets_per_frame + (e.y >> p.bucket_log2);
            cnt = ld_cg(slot_cnt(p, e.x));
        }
        const bool ok = act && d < p.occ_cap;
        if (act && !ok) set_status(p.hdr, MMBEV_DEV_BOUNDS);
        // the voxels' segments: a block-wide exclusive scan of the counts and
        // one atomicAdd on the global total per chunk
        const uint32_t c = ok ? cnt : 0u;
        uint32_t inc = c;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const uint32_t x = __shfl_up_sync(0xFFFFFFFFu, inc, o);
            if (lane >= o) inc += x;
        }
        if (lane == 31) s_seg[warp] = inc;
        __syncthreads();
        if (t == 0) {
            uint32_t run = 0;
            for (int w = 0; w < kCompactThreads / 32; ++w) {
                const uint32_t x = s_seg[w];
                s_seg[w] = run;
                run += x;
            }
            s_segbase = run ? atomicAdd(&p.hdr->seg_total, run) : 0u;
        }
        __syncthreads();
        const uint32_t segoff = s_segbase + s_seg[warp] + inc - c;
        __syncthreads();
        // warp-aggregated bucket count: one atomicAdd per distinct bucket
        const uint32_t am = __ballot_sync(0xFFFFFFFFu, ok);
        uint32_t grp = 1u << lane;
        if (ok) grp = __match_any_sync(am, bk);
        const int leader = __ffs(grp) - 1;
        uint32_t pos = 0;
        if (ok && lane == leader)
            pos = (uint32_t)atomicAdd(&p.bcnt[bk], (unsigned long long)__popc(grp));
        pos = __shfl_sync(0xFFFFFFFFu, pos, leader) + __popc(grp & ((1u << lane) - 1u));
        // and into its scan chunk (kScanChunk consecutive buckets of a frame)
        const uint32_t ch = e.z * p.scan_chunks + ((e.y >> p.bucket_log2) / kScanChunk);
        uint32_t cgrp = 1u << lane;
        if (ok) cgrp = __match_any_sync(am, ch);
        if (ok && lane == __ffs(cgrp) - 1) atomicAdd(&p.ctot[ch], (uint32_t)__popc(cgrp));
        // slots with more than kLightMax points, for the finalize stage's heavy
        // role (counts sum to at most occ_cap points: the lists have room)
        const bool heavy = ok && cnt > kLightMax && cnt <= kHugeMin;
        const uint32_t hm = __ballot_sync(0xFFFFFFFFu, heavy);
        if (hm) {
            const int hl = __ffs(hm) - 1;
            uint32_t hb = 0;
            if (lane == hl) hb = atomicAdd(&p.hdr->num_heavy, (uint32_t)__popc(hm));
            hb = __shfl_sync(0xFFFFFFFFu, hb, hl) + __popc(hm & ((1u << lane) - 1u));
            if (heavy) {
                if (hb < p.occ_cap / (kLightMax + 1) + 1) p.heavy[hb] = e.x;
                else set_status(p.hdr, MMBEV_DEV_BOUNDS);
            }
        }
        if (ok && cnt > kHugeMin) {   // rare
            const uint32_t hu = atomicAdd(&p.hdr->num_huge, 1u);
            if (hu < p.occ_cap / (kHugeMin + 1) + 1) p.huge[hu] = e.x;
            else set_status(p.hdr, MMBEV_DEV_BOUNDS);
        }
        if (ok) {
            *slot_seg(p, e.x) = segoff;
            p.occ[d] = e.x;
            p.d_lin[d] = e.y;
            p.d_bucket[d] = bk;
            p.d_pos[d] = pos;
            const uint32_t fo = e.z - s_fmin;
            if (fo < (uint32_t)kFrameWin) atomicAdd(&s_fcnt[fo], 1u);
            else atomicAdd(&p.frame_u[e.z], 1u);
        }
    }
    __syncthreads();
    if (t < kFrameWin && s_fcnt[t]) atomicAdd(&p.frame_u[s_fmin + t], s_fcnt[t]);
}

__global__ void __launch_bounds__(kThreads, kBlocksPerSm) k_scatter_points(Params p) {
    __shared__ Lists L;
    __shared__ uint32_t s_part[kThreads / 32];
    pdl_wait();
    // frames with more voxels than max_voxels need each voxel's minimum ROI
    // rank (the cap keeps the smallest (rank, lin)); others never read it
    int capped = 0;
    for (int f = threadIdx.x; f < p.num_frames; f += blockDim.x)
        capped |= ld_cg(&p.frame_u[f]) > (uint32_t)p.max_voxels;
    capped = __syncthreads_or(capped);
    const uint32_t M = lists_scan(p, L, s_part);
    const uint32_t cap = min(ld_cg(&p.hdr->seg_total), p.occ_cap);  // seg holds N entries
    const uint32_t gs = gridDim.x * blockDim.x;
    for (uint32_t i = blockIdx.x * blockDim.x + threadIdx.x; i < M; i += gs) {
        const size_t e = list_entry(p, L, i);
        const uint2 hs = p.rs[e];
        if (hs.x == kUnset) continue;
        const uint32_t pos = p.plist[e].z;
        const uint32_t at = ld_cg(slot_seg(p, hs.x)) + hs.y;
        if (at < cap) p.seg[at] = pos;
        else set_status(p.hdr, MMBEV_DEV_BOUNDS);
        if (capped) {
            const uint32_t f = p.plist[e].y;
            if (f < (uint32_t)p.num_frames && ld_cg(&p.frame_u[f]) > (uint32_t)p.max_voxels &&
                pos < p.rec_cap)
                atomicMax(slot_rank(p, hs.x), 0xFFFFFFFFu - p.records[2 * (size_t)pos + 1].y);
        }
    }
}

}  // namespace

uint32_t insert_blocks(int num_sms) { return (uint32_t)num_sms * kBlocksPerSm; }

cudaError_t launch_insert(const Params& p, bool pdl, cudaStream_t st) {
    return launch_k(k_insert, dim3(p.ins_blocks), dim3(kThreads), 0, st, pdl, p);
}

cudaError_t launch_compact(const Params& p, bool pdl, cudaStream_t st) {
    return launch_k(k_compact, dim3(p.ins_blocks), dim3(kCompactThreads), 0, st, pdl, p);
}

cudaError_t launch_scatter_points(const Params& p, bool pdl, cudaStream_t st) {
    return launch_k(k_scatter_points, dim3(p.ins_blocks), dim3(kThreads), 0, st, pdl, p);
}

}  // namespace mmbev
