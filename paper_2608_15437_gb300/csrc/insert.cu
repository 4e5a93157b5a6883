// Stage 2: voxel hash insert and dedup (S3 of the path; Alg. 1 "Voxelize"),
// stage 3: the occupied-voxel list, stage 4: per-voxel point lists.
//
// Insert. Every block owns a contiguous range of 32-point regions; each warp
// takes one region's kept-point records (at most 32) at a time, with no block
// barrier in the loop:
//   1. lanes holding the same voxel key are grouped with __match_any_sync
//      (all later warp collectives run on the full warp);
//   2. the group leader reads the key's home slot (key, minimum rank) in one
//      round trip; a matching key means found, an empty slot is claimed with
//      atomicCAS, another key moves on to the next slot (linear probing, at
//      most H probes). It lowers the slot's minimum ROI rank (stored as
//      0xFFFFFFFF - rank, so an all-zero slot is empty) with a
//      fire-and-forget atomicMax only when the group improves it, and adds
//      the group's size to the slot's point count with one atomicAdd whose
//      old value numbers the group's points;
//   3. each lane stores {slot, arrival number} at its record position.
//   A leader that created the slot appends {slot, lin, frame} to its block's
//   own sub-list (one shared-memory atomic per warp), so no global counter
//   is touched. No point ever waits on another point's insertion: the
//   voxel's first K points are chosen later, from the complete list.
// Compact. One block per insert block copies that block's sub-list into the
// dense occupied-voxel list at the sum of the earlier blocks' counts, counts
// every new voxel into its frame and into its ordering bucket (warp-
// aggregated, recording its position in the bucket), and reserves the
// voxel's segment of `seg` (one atomicAdd per block chunk), written into the
// slot.
// Scatter points. Every record's position goes to seg[slot segment +
// arrival number], so each voxel's points end up contiguous.
#include "mmbev_internal.cuh"

namespace mmbev {
namespace {

constexpr int kThreads = 256;
constexpr int kBlocksPerSm = 6;
constexpr int kFrameWin = 64;

__global__ void __launch_bounds__(kThreads, kBlocksPerSm) k_insert(Params p) {
    __shared__ uint32_t s_nnew;
    pdl_wait();
    pdl_trigger();
    const int t = threadIdx.x, lane = t & 31, warp = t >> 5;
    if (t == 0) s_nnew = 0;
    __syncthreads();
    const uint32_t RG = p.num_regions;
    const uint32_t rb = (uint32_t)((uint64_t)blockIdx.x * RG / gridDim.x);
    const uint32_t re = (uint32_t)((uint64_t)(blockIdx.x + 1) * RG / gridDim.x);
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
    uint4* sub = p.newlist + (size_t)rb * kRegion;
    for (uint32_t g = rb + (uint32_t)warp; g < re; g += (uint32_t)nwarps) {
        const uint32_t n = min(ld_cg(&p.reg_cnt[g]), (uint32_t)kRegion);
        if (n == 0) continue;
        const uint32_t r = g * (uint32_t)kRegion + lane;
        const uint4* rec = p.records;
        uint2* rs = p.rec_slot;
        const bool act = (uint32_t)lane < n;
        const uint32_t am = __ballot_sync(0xFFFFFFFFu, act);
        uint4 a = make_uint4(0u, 0u, 0u, 0u);
        unsigned long long key = ~0ull;
        uint32_t grp = 1u << lane;
        if (act) {
            a = __ldcs(rec + 2 * r);   // lin, frame, rank, x'
            key = ((unsigned long long)a.y << 32) | a.x;
            grp = __match_any_sync(am, key);
        }
        const int leader = __ffs(grp) - 1;
        uint32_t gmin_rank = a.z;
        if (__any_sync(0xFFFFFFFFu, grp != (1u << lane))) {
            // some voxel appears more than once in this warp
            for (int l = 0; l < 32; ++l) {
                const uint32_t rl = __shfl_sync(0xFFFFFFFFu, a.z, l);
                if ((grp >> l) & 1u) gmin_rank = rl < gmin_rank ? rl : gmin_rank;
            }
        }
        bool created = false;
        uint32_t h = kUnset, base = 0;
        if (act && lane == leader) {
            const unsigned long long key1 = key + 1ull;
            h = slot_home(mask, key1);
            uint4 s0 = make_uint4(0u, 0u, 0u, 0u);
            bool done = false;
            for (uint32_t probe = 0; probe <= mask; ++probe) {
                s0 = __ldcg(reinterpret_cast<const uint4*>(slot_key(p, h)));  // key, rank, cnt
                const unsigned long long cur = ((unsigned long long)s0.y << 32) | s0.x;
                if (cur == key1) { done = true; break; }
                if (cur == 0ull) {
                    const unsigned long long old = atomicCAS(slot_key(p, h), 0ull, key1);
                    if (old == 0ull) { created = true; done = true; s0.z = 0u; break; }
                    if (old == key1) { done = true; s0.z = 0u; break; }
                }
                h = (h + 1u) & mask;
            }
            if (!done) {
                set_status(p.hdr, MMBEV_DEV_TABLE_FULL);
                h = kUnset;
            } else {
                const uint32_t enc = 0xFFFFFFFFu - gmin_rank;
                if (enc > s0.z) atomicMax(slot_rank(p, h), enc);
                base = atomicAdd(slot_cnt(p, h), (uint32_t)__popc(grp));
            }
        }
        h = __shfl_sync(0xFFFFFFFFu, h, leader);
        base = __shfl_sync(0xFFFFFFFFu, base, leader);
        if (act) rs[r] = make_uint2(h, base + __popc(grp & ((1u << lane) - 1u)));
        // leaders of new slots append to this block's sub-list
        const uint32_t cm = __ballot_sync(0xFFFFFFFFu, created);
        if (cm) {
            uint32_t wbase = 0;
            if (lane == __ffs(cm) - 1) wbase = atomicAdd(&s_nnew, (uint32_t)__popc(cm));
            wbase = __shfl_sync(0xFFFFFFFFu, wbase, __ffs(cm) - 1);
            if (created) sub[wbase + __popc(cm & ((1u << lane) - 1u))] = make_uint4(h, a.x, a.y, 0u);
        }
    }
    __syncthreads();
    if (t == 0) p.blockcount[blockIdx.x] = s_nnew;
}

__global__ void __launch_bounds__(kThreads) k_compact(Params p) {
    __shared__ uint32_t s_red[kThreads / 32];
    __shared__ uint32_t s_seg[kThreads / 32];
    __shared__ uint32_t s_base, s_segbase;
    __shared__ uint32_t s_fcnt[kFrameWin];
    __shared__ uint32_t s_fmin;
    pdl_wait();
    pdl_trigger();
    const int t = threadIdx.x, lane = t & 31, warp = t >> 5;
    const uint32_t b = blockIdx.x;
    // this block's place: the sum of the earlier blocks' counts
    uint32_t part = 0;
    for (uint32_t i = t; i < b; i += kThreads) part += p.blockcount[i];
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) part += __shfl_xor_sync(0xFFFFFFFFu, part, o);
    if (lane == 0) s_red[warp] = part;
    if (t < kFrameWin) s_fcnt[t] = 0;
    const uint32_t rb = (uint32_t)((uint64_t)b * p.num_regions / p.ins_blocks);
    const uint4* sub = p.newlist + (size_t)rb * kRegion;
    const uint32_t n = p.blockcount[b];
    if (t == 0) s_fmin = n ? sub[0].z : 0u;
    __syncthreads();
    if (t == 0) {
        uint32_t s = 0;
        for (int w = 0; w < kThreads / 32; ++w) s += s_red[w];
        s_base = s;
        if (b == p.ins_blocks - 1) p.hdr->num_occ = s + n;
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

__global__ void __launch_bounds__(kThreads) k_scatter_points(Params p) {
    pdl_wait();
    pdl_trigger();
    const uint32_t cap = ld_cg(&p.hdr->seg_total);
    const size_t npos = (size_t)p.num_regions * kRegion;
    const size_t gs = (size_t)gridDim.x * blockDim.x;
    for (size_t r = (size_t)blockIdx.x * blockDim.x + threadIdx.x; r < npos; r += gs) {
        const uint32_t n = ld_cg(&p.reg_cnt[r / kRegion]);
        if ((uint32_t)(r % kRegion) >= n) continue;
        const uint2 hs = p.rec_slot[r];
        if (hs.x == kUnset) continue;
        const uint32_t at = ld_cg(slot_seg(p, hs.x)) + hs.y;
        if (at < cap) p.seg[at] = (uint32_t)r;
        else set_status(p.hdr, MMBEV_DEV_BOUNDS);
    }
}

}  // namespace

uint32_t insert_blocks(int num_sms) { return (uint32_t)num_sms * kBlocksPerSm; }

cudaError_t launch_insert(const Params& p, bool pdl, cudaStream_t st) {
    return launch_k(k_insert, dim3(p.ins_blocks), dim3(kThreads), 0, st, pdl, p);
}

cudaError_t launch_compact(const Params& p, bool pdl, cudaStream_t st) {
    return launch_k(k_compact, dim3(p.ins_blocks), dim3(kThreads), 0, st, pdl, p);
}

cudaError_t launch_scatter_points(const Params& p, bool pdl, cudaStream_t st) {
    return launch_k(k_scatter_points, dim3(p.ins_blocks), dim3(kThreads), 0, st, pdl, p);
}

}  // namespace mmbev
