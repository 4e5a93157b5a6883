// Stage 2: voxel hash insert and dedup (S3 of the path; Alg. 1 "Voxelize"),
// stage 3: the occupied-voxel list, stage 4: per-voxel point lists.
//
// Insert. One block per 2048-point tile; its warps take the tile's kept-point
// records in batches of 32 (the next batch's records load while the current
// batch is inserted), with no block barrier in the loop:
//   1. lanes holding the same voxel key are grouped with __match_any_sync
//      (all later warp collectives run on the full warp);
//   2. the group leader finds the key's slot from its home slot (linear
//      probing, at most H probes): a matching key means found, an empty slot
//      is claimed with atomicCAS; it adds the group's size to the slot's
//      point count with one atomicAdd whose old value numbers the group's
//      points (an all-zero slot is empty);
//   3. each lane stores {slot, arrival number} at its record position.
//   A leader that created the slot appends {slot, lin, frame} to its tile's
//   sub-list (one shared-memory atomic per warp). No point ever waits on
//   another point's insertion: the voxel's first K points are chosen later,
//   from the complete list.
// Compact. One block per tile copies the tile's sub-list into the dense
// occupied-voxel list at a place taken with one atomicAdd (the list's order
// is immaterial), counts every new voxel into its frame and into its
// ordering bucket (warp-aggregated, recording its position in the bucket),
// and reserves the voxel's segment of `seg` (one atomicAdd per block chunk),
// written into the slot.
// Scatter points. Every record's position goes to seg[slot segment +
// arrival number], so each voxel's points end up contiguous.
#include "mmbev_internal.cuh"

namespace mmbev {
namespace {

constexpr int kThreads = 256;
constexpr int kBlocksPerSm = 8;
constexpr int kFrameWin = 64;
constexpr uint32_t kFull = 0xFFFFFFFFu;

// One block per 2048-point tile. The tile's 64 region counts are scanned in
// shared memory; the tile's kept records are then taken in batches of 32 by
// the block's warps in turn (record j of the tile lies in the region whose
// range [excl, incl) holds j, found by a six-step binary search).
struct TileScan {
    uint32_t incl[kTile / kRegion];
    uint32_t excl[kTile / kRegion];
};

// Threads 0..63 read the counts; every thread must call it (one barrier).
// Returns the tile's kept records.
__device__ __forceinline__ uint32_t tile_scan(const Params& p, uint32_t tile, TileScan& ts,
                                              uint32_t* s_part) {
    const int t = threadIdx.x, lane = t & 31;
    uint32_t n = 0, v = 0;
    if (t < kTile / kRegion) {
        n = min(ld_cg(&p.reg_cnt[tile * (kTile / kRegion) + t]), (uint32_t)kRegion);
        v = n;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const uint32_t x = __shfl_up_sync(kFull, v, o);
            if (lane >= o) v += x;
        }
        if (lane == 31) s_part[t >> 5] = v;
    }
    __syncthreads();
    if (t < kTile / kRegion) {
        if (t >= 32) v += s_part[0];
        ts.incl[t] = v;
        ts.excl[t] = v - n;
    }
    __syncthreads();
    return ts.incl[kTile / kRegion - 1];
}

__device__ __forceinline__ uint32_t tile_item_pos(const TileScan& ts, uint32_t tile, uint32_t j) {
    int l = 0;  // regions whose range ends at or before j
#pragma unroll
    for (int step = 32; step >= 1; step >>= 1)
        if (l + step <= kTile / kRegion && ts.incl[l + step - 1] <= j) l += step;
    if (l > kTile / kRegion - 1) l = kTile / kRegion - 1;
    return (tile * (kTile / kRegion) + (uint32_t)l) * kRegion + (j - ts.excl[l]);
}

__global__ void __launch_bounds__(kThreads, kBlocksPerSm) k_insert(Params p) {
    __shared__ TileScan ts;
    __shared__ uint32_t s_part[2];
    __shared__ uint32_t s_nnew;
    pdl_wait();
    pdl_trigger();
    const int t = threadIdx.x, lane = t & 31, warp = t >> 5;
    const uint32_t tile = blockIdx.x;
    if (t == 0) s_nnew = 0;
    const uint32_t total = tile_scan(p, tile, ts, s_part);
    // slots in use: a power of two >= 1.25 x the call's kept points
    uint32_t lg = 10;
    if (p.table_log2_fixed > 0) {
        lg = (uint32_t)p.table_log2_fixed;
    } else {
        const uint64_t need = (uint64_t)ld_cg(&p.hdr->num_rec) * 5 / 4;
        while (lg < p.table_log2 && (1ull << lg) < need) ++lg;
    }
    const uint32_t mask = (uint32_t)((1ull << lg) - 1ull);
    const int nwarps = kThreads / 32;
    const uint32_t lt = (1u << lane) - 1u;
    // the tile's sub-list of created voxels: room for every record of the tile
    uint4* sub = p.newlist + (size_t)tile * kTile;
    // batch j0 is processed while the warp's next batch's records load
    uint32_t j = (uint32_t)warp * 32u + lane;
    bool act = j < total;
    uint32_t pos = act ? tile_item_pos(ts, tile, j) : 0u;
    uint2 a = act ? __ldcs(p.keys + pos) : make_uint2(0u, 0u);   // lin, frame
    for (uint32_t j0 = (uint32_t)warp * 32u; j0 < total; j0 += nwarps * 32u) {
        const uint32_t jn = j0 + nwarps * 32u + lane;
        const bool actn = jn < total;
        const uint32_t posn = actn ? tile_item_pos(ts, tile, jn) : 0u;
        const uint2 an = actn ? __ldcs(p.keys + posn) : make_uint2(0u, 0u);

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
        if (act) p.rec_slot[pos] = make_uint2(h, base + __popc(grp & lt));
        // leaders of new slots append to the tile's sub-list
        const uint32_t cm = __ballot_sync(kFull, created);
        if (cm) {
            uint32_t wbase = 0;
            if (lane == __ffs(cm) - 1) wbase = atomicAdd(&s_nnew, (uint32_t)__popc(cm));
            wbase = __shfl_sync(kFull, wbase, __ffs(cm) - 1);
            if (created) sub[wbase + __popc(cm & lt)] = make_uint4(h, a.x, a.y, 0u);
        }
        a = an;
        pos = posn;
        act = actn;
    }
    __syncthreads();
    if (t == 0) p.blockcount[tile] = s_nnew;
}

__global__ void __launch_bounds__(kThreads) k_compact(Params p) {
    __shared__ uint32_t s_seg[kThreads / 32];
    __shared__ uint32_t s_base, s_segbase;
    __shared__ uint32_t s_fcnt[kFrameWin];
    __shared__ uint32_t s_fmin;
    pdl_wait();
    pdl_trigger();
    const int t = threadIdx.x, lane = t & 31, warp = t >> 5;
    const uint32_t b = blockIdx.x;
    const uint4* sub = p.newlist + (size_t)b * kTile;
    const uint32_t n = p.blockcount[b];
    if (n == 0) return;
    if (t < kFrameWin) s_fcnt[t] = 0;
    // this tile's place in the occupied-voxel list (order is immaterial)
    if (t == 0) {
        s_fmin = sub[0].z;
        s_base = atomicAdd(&p.hdr->num_occ, n);
    }
    __syncthreads();
    const uint32_t base = s_base;
    for (uint32_t i0 = 0; i0 < n; i0 += kThreads) {
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
            for (int w = 0; w < kThreads / 32; ++w) {
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
    __shared__ TileScan ts;
    __shared__ uint32_t s_part[2];
    pdl_wait();
    pdl_trigger();
    const uint32_t tile = blockIdx.x;
    // frames with more voxels than max_voxels need each voxel's minimum ROI
    // rank (the cap keeps the smallest (rank, lin)); others never read it
    int capped = 0;
    for (int f = threadIdx.x; f < p.num_frames; f += blockDim.x)
        capped |= ld_cg(&p.frame_u[f]) > (uint32_t)p.max_voxels;
    capped = __syncthreads_or(capped);
    const uint32_t total = tile_scan(p, tile, ts, s_part);
    const uint32_t cap = min(ld_cg(&p.hdr->seg_total), p.occ_cap);  // seg holds N entries
    for (uint32_t j = threadIdx.x; j < total; j += blockDim.x) {
        const uint32_t pos = tile_item_pos(ts, tile, j);
        const uint2 hs = p.rec_slot[pos];
        if (hs.x == kUnset) continue;
        const uint32_t at = ld_cg(slot_seg(p, hs.x)) + hs.y;
        if (at < cap) p.seg[at] = pos;
        else set_status(p.hdr, MMBEV_DEV_BOUNDS);
        if (capped) {
            const uint32_t f = p.keys[pos].y;
            if (ld_cg(&p.frame_u[f]) > (uint32_t)p.max_voxels)
                atomicMax(slot_rank(p, hs.x), 0xFFFFFFFFu - p.records[2 * (size_t)pos + 1].y);
        }
    }
}

}  // namespace

cudaError_t launch_insert(const Params& p, bool pdl, cudaStream_t st) {
    const uint32_t tiles = p.num_regions / (kTile / kRegion);
    if (tiles == 0) return cudaSuccess;
    return launch_k(k_insert, dim3(tiles), dim3(kThreads), 0, st, pdl, p);
}

cudaError_t launch_compact(const Params& p, bool pdl, cudaStream_t st) {
    const uint32_t tiles = p.num_regions / (kTile / kRegion);
    if (tiles == 0) return cudaSuccess;
    return launch_k(k_compact, dim3(tiles), dim3(kThreads), 0, st, pdl, p);
}

cudaError_t launch_scatter_points(const Params& p, bool pdl, cudaStream_t st) {
    const uint32_t tiles = p.num_regions / (kTile / kRegion);
    if (tiles == 0) return cudaSuccess;
    return launch_k(k_scatter_points, dim3(tiles), dim3(kThreads), 0, st, pdl, p);
}

}  // namespace mmbev
