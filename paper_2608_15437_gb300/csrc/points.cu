// Stage 1: the point pass (S1 + S2 + S3 of the path).
//
// One block takes a tile of 2048 consecutive points:
//   A. loads the tile's 40 KB of float32 AoS points into shared memory with
//      coalesced 16-byte streaming loads, stages the tile's sweep transforms;
//   B. per point: Eq. 6 motion compensation, range crop, Alg. 1 inside-ROI
//      test (coarse candidate mask, then the exact rotated-box test in rank
//      order; the first hit is the point's rank), voxel index;
//   C. ballot/popc compaction of the kept points into a shared queue that
//      preserves input order;
//   D. hash insert of the queue: lanes with equal keys are grouped with
//      __match_any_sync; the group leader probes / claims the slot and lowers
//      the slot's minimum rank once for the group; every lane then inserts its
//      point index into the slot's bounded "K smallest indices" list;
//   E. one atomicAdd per block appends the block's new slots to the
//      occupied-slot list; per-frame voxel counts are block-aggregated too.
#include "mmbev_internal.cuh"

namespace mmbev {
namespace {

constexpr int kTfStage = 64;   // sweeps staged in smem per tile
constexpr int kFrameCnt = 32;  // frames counted in smem per tile
constexpr int kWarps = kPtsThreads / 32;

struct QItem {
    unsigned long long key;
    uint32_t idx;
    uint32_t rank;
};
static_assert(kTile * sizeof(QItem) + kTile * sizeof(uint32_t) <= kTile * 5 * sizeof(float),
              "queue and new-slot list must fit in the point tile");

// Sweep of global point index i: largest s with off[s] <= i (off nondecreasing).
__device__ __forceinline__ int find_sweep(const int64_t* off, int nsweeps, int64_t i) {
    int lo = 0, hi = nsweeps;  // off[lo] <= i < off[hi]
    while (hi - lo > 1) {
        const int mid = (lo + hi) >> 1;
        if (off[mid] <= i) lo = mid; else hi = mid;
    }
    return lo;
}

// Claim or find the slot of key+1 by linear probing; at most H probes.
// Returns the slot, sets *is_new when this call claimed it; 0xFFFFFFFF when
// the table is full.
__device__ __forceinline__ uint32_t table_insert(const Params& p, unsigned long long key1,
                                                 bool* is_new) {
    const uint32_t mask = (uint32_t)((1ull << p.table_log2) - 1ull);
    uint32_t h = (uint32_t)mix64(key1) & mask;
    *is_new = false;
    for (uint64_t probe = 0; probe <= mask; ++probe) {
        unsigned long long* kp = slot_key(p, h);
        const unsigned long long cur = ld_cg(kp);
        if (cur == key1) return h;
        if (cur == 0ull) {
            const unsigned long long old = atomicCAS(kp, 0ull, key1);
            if (old == 0ull) { *is_new = true; return h; }
            if (old == key1) return h;
        }
        h = (h + 1u) & mask;
    }
    return kUnset;
}

// Insert v = ~index into the slot's sorted list of the K largest values
// (= the K smallest point indices). Levels only ever grow, so a level read
// as >= v stays >= v and can be skipped; each atomicMax keeps the larger of
// (level, v) and carries the smaller one down; an empty level (0) ends it.
__device__ __forceinline__ void topk_insert(uint32_t* tk, uint32_t v, int K) {
    int j = 0;
    while (j < K) {
        // One round trip reads up to 12 levels.
        uint32_t lv[12];
        const int nread = (K - j) < 12 ? (K - j) : 12;
#pragma unroll
        for (int c = 0; c < 12; ++c) lv[c] = c < nread ? ld_cg(tk + j + c) : 0u;
        int first = nread;
#pragma unroll
        for (int c = 11; c >= 0; --c)
            if (c < nread && lv[c] < v) first = c;
        j += first;
        if (first < nread) break;
    }
    for (; j < K; ++j) {
        const uint32_t old = atomicMax(tk + j, v);
        if (old == 0u) return;
        v = old < v ? old : v;
    }
}

template <bool kClassify>
__global__ void __launch_bounds__(kPtsThreads)
k_points(Params p) {
    __shared__ __align__(16) float s_pts[kTile * 5];
    __shared__ __align__(16) float s_tf[kTfStage][12];
    __shared__ int64_t s_soff[kTfStage + 1];
    __shared__ int32_t s_sfr[kTfStage];
    __shared__ int32_t s_r0[kTfStage];
    __shared__ uint32_t s_wcnt[kPtsPerThread * kWarps];
    __shared__ uint32_t s_fcnt[kFrameCnt];
    __shared__ int s_slo, s_nst;
    __shared__ uint32_t s_nq, s_nnew, s_occ_base;

    const int t = threadIdx.x, lane = t & 31, warp = t >> 5;
    const int64_t tile_base = (int64_t)blockIdx.x * kTile;
    const int64_t rem = p.num_points - tile_base;
    const int n = rem < (int64_t)kTile ? (int)rem : kTile;
    if (n <= 0) return;

    // ---- A. stage points and sweep metadata
    {
        const float* src = p.points + tile_base * 5;
        const int nf = n * 5;
        const int n4 = nf >> 2;
        const float4* src4 = reinterpret_cast<const float4*>(src);
        float4* dst4 = reinterpret_cast<float4*>(s_pts);
        for (int i = t; i < n4; i += kPtsThreads) dst4[i] = __ldcs(src4 + i);
        for (int i = (n4 << 2) + t; i < nf; i += kPtsThreads) s_pts[i] = __ldcs(src + i);
    }
    if (t == 0) {
        const int slo = find_sweep(p.sweep_off, p.num_sweeps, tile_base);
        const int shi = find_sweep(p.sweep_off, p.num_sweeps, tile_base + n - 1);
        s_slo = slo;
        s_nst = shi - slo + 1;
        s_nq = 0;
        s_nnew = 0;
    }
    if (t < kFrameCnt) s_fcnt[t] = 0u;
    __syncthreads();
    const int slo = s_slo, nst = s_nst;
    const bool staged = nst <= kTfStage;
    if (staged) {
        for (int i = t; i < nst * 12; i += kPtsThreads) {
            const int k = i / 12, c = i % 12;
            s_tf[k][c] = __ldg(p.sweep_tf + (size_t)(slo + k) * 16 + c);
        }
        for (int i = t; i <= nst; i += kPtsThreads) s_soff[i] = p.sweep_off[slo + i];
        for (int i = t; i < nst; i += kPtsThreads) {
            const int f = p.sweep_frame[slo + i];
            s_sfr[i] = f;
            s_r0[i] = p.frame_roi_off[f];
        }
    }
    __syncthreads();
    const int f_first = staged ? s_sfr[0] : 0;

    // ---- B. per point
    const int G = p.coarse, W = p.mask_words;
    unsigned long long key[kPtsPerThread];
    uint32_t rank[kPtsPerThread];
    bool valid[kPtsPerThread];
#pragma unroll
    for (int k = 0; k < kPtsPerThread; ++k) {
        const int j = t + k * kPtsThreads;
        valid[k] = false;
        key[k] = 0ull;
        rank[k] = 0u;
        if (j >= n) continue;
        const int64_t idx = tile_base + j;
        const float* q = s_pts + 5 * j;
        int sl;
        const float* T;
        int f, r0;
        float Tg[12];
        if (staged) {
            sl = 0;
            while (s_soff[sl + 1] <= idx) ++sl;
            T = s_tf[sl];
            f = s_sfr[sl];
            r0 = s_r0[sl];
        } else {
            const int s = find_sweep(p.sweep_off, p.num_sweeps, idx);
#pragma unroll
            for (int c = 0; c < 12; ++c) Tg[c] = __ldg(p.sweep_tf + (size_t)s * 16 + c);
            T = Tg;
            f = p.sweep_frame[s];
            r0 = p.frame_roi_off[f];
        }
        float x, y, z;
        compensate(T, q[0], q[1], q[2], x, y, z);
        if (kClassify) {
            p.cls_xyz[idx * 3 + 0] = x;
            p.cls_xyz[idx * 3 + 1] = y;
            p.cls_xyz[idx * 3 + 2] = z;
        }
        bool ok = (p.rmin[0] <= x) && (x < p.rmax[0]) && (p.rmin[1] <= y) && (y < p.rmax[1]) &&
                  (p.rmin[2] <= z) && (z < p.rmax[2]);
        int r_hit = -1;
        if (ok) {
            int gx = (int)__fmul_rn(__fsub_rn(x, p.rmin[0]), p.coarse_inv[0]);
            int gy = (int)__fmul_rn(__fsub_rn(y, p.rmin[1]), p.coarse_inv[1]);
            gx = min(max(gx, 0), G - 1);
            gy = min(max(gy, 0), G - 1);
            const uint32_t* mw = p.masks + ((size_t)f * G * G + (size_t)gy * G + gx) * W;
            for (int w = 0; w < W && r_hit < 0; ++w) {
                uint32_t bits = __ldg(mw + w);
                while (bits) {
                    const int b = __ffs(bits) - 1;
                    bits &= bits - 1u;
                    const int r = w * 32 + b;
                    const RoiPrep rp = p.roi_prep[r0 + r];
                    if (roi_contains(rp, x, y)) { r_hit = r; break; }
                }
            }
        }
        uint32_t lin = 0;
        if (r_hit >= 0) {
            const uint32_t cx = __float2uint_rz(__fdiv_rn(__fsub_rn(x, p.rmin[0]), p.vs[0]));
            const uint32_t cy = __float2uint_rz(__fdiv_rn(__fsub_rn(y, p.rmin[1]), p.vs[1]));
            const uint32_t cz = __float2uint_rz(__fdiv_rn(__fsub_rn(z, p.rmin[2]), p.vs[2]));
            if (cx < p.dims[0] && cy < p.dims[1] && cz < p.dims[2]) {
                lin = (cz * p.dims[1] + cy) * p.dims[0] + cx;
                valid[k] = true;
                rank[k] = (uint32_t)r_hit;
                key[k] = ((unsigned long long)(uint32_t)f << 32) | lin;
            }
        }
        if (kClassify) {
            p.cls_lin[idx] = valid[k] ? (int64_t)lin : (int64_t)-1;
            p.cls_rank[idx] = valid[k] ? r_hit : -1;
        }
    }
    if (kClassify) return;

    // ---- C. order-preserving compaction into the shared queue
    uint32_t ballots[kPtsPerThread];
#pragma unroll
    for (int k = 0; k < kPtsPerThread; ++k) {
        ballots[k] = __ballot_sync(0xFFFFFFFFu, valid[k]);
        if (lane == 0) s_wcnt[k * kWarps + warp] = __popc(ballots[k]);
    }
    __syncthreads();
    if (warp == 0) {
        // exclusive scan of 64 counts, two per lane, in (k, warp) order
        const uint32_t a = s_wcnt[2 * lane], b = s_wcnt[2 * lane + 1];
        uint32_t s = a + b;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const uint32_t v = __shfl_up_sync(0xFFFFFFFFu, s, o);
            if (lane >= o) s += v;
        }
        const uint32_t excl = s - (a + b);
        s_wcnt[2 * lane] = excl;
        s_wcnt[2 * lane + 1] = excl + a;
        if (lane == 31) s_nq = s;
    }
    __syncthreads();
    QItem* queue = reinterpret_cast<QItem*>(s_pts);
    uint32_t* new_slots = reinterpret_cast<uint32_t*>(queue + kTile);
    const uint32_t lt = (1u << lane) - 1u;
#pragma unroll
    for (int k = 0; k < kPtsPerThread; ++k) {
        if (valid[k]) {
            const uint32_t pos = s_wcnt[k * kWarps + warp] + __popc(ballots[k] & lt);
            QItem it;
            it.key = key[k];
            it.idx = (uint32_t)(tile_base + t + k * kPtsThreads);
            it.rank = rank[k];
            queue[pos] = it;
        }
    }
    __syncthreads();

    // ---- D. hash insert
    const uint32_t nq = s_nq;
    for (uint32_t base = (uint32_t)warp * 32u; base < nq; base += kPtsThreads) {
        const uint32_t i = base + lane;
        const bool act = i < nq;
        const uint32_t am = __ballot_sync(0xFFFFFFFFu, act);
        if (!act) continue;
        const QItem it = queue[i];
        const uint32_t grp = __match_any_sync(am, it.key);
        const int leader = __ffs(grp) - 1;
        const uint32_t gmin = __reduce_min_sync(grp, it.rank);
        uint32_t h = kUnset;
        if (lane == leader) {
            bool is_new = false;
            h = table_insert(p, it.key + 1ull, &is_new);
            if (h == kUnset) {
                set_status(p.hdr, MMBEV_DEV_TABLE_FULL);
            } else {
                uint32_t* rk = slot_rank(p, h);
                const uint32_t enc = 0xFFFFFFFFu - gmin;
                if (ld_cg(rk) < enc) atomicMax(rk, enc);
                if (is_new) {
                    const uint32_t slot_i = atomicAdd(&s_nnew, 1u);
                    new_slots[slot_i] = h;
                    const uint32_t fo = (uint32_t)(it.key >> 32) - (uint32_t)f_first;
                    if (staged && fo < (uint32_t)kFrameCnt) atomicAdd(&s_fcnt[fo], 1u);
                    else atomicAdd(&p.frame_u[it.key >> 32], 1u);
                }
            }
        }
        h = __shfl_sync(grp, h, leader);
        if (h != kUnset) topk_insert(slot_topk(p, h), ~it.idx, p.K);
    }
    __syncthreads();

    // ---- E. publish new slots and per-frame counts
    const uint32_t nnew = s_nnew;
    if (t == 0 && nnew > 0) s_occ_base = atomicAdd(&p.hdr->num_occ, nnew);
    if (staged && t < kFrameCnt && s_fcnt[t] > 0) atomicAdd(&p.frame_u[f_first + t], s_fcnt[t]);
    __syncthreads();
    const uint32_t ob = s_occ_base;
    for (uint32_t i = t; i < nnew; i += kPtsThreads) {
        if (ob + i < p.occ_cap) p.occ[ob + i] = new_slots[i];
        else set_status(p.hdr, MMBEV_DEV_BOUNDS);
    }
}

}  // namespace

cudaError_t launch_points(const Params& p, bool classify_only, cudaStream_t st) {
    if (p.num_points <= 0) return cudaSuccess;
    const int64_t blocks = (p.num_points + kTile - 1) / kTile;
    if (classify_only) k_points<true><<<(unsigned)blocks, kPtsThreads, 0, st>>>(p);
    else k_points<false><<<(unsigned)blocks, kPtsThreads, 0, st>>>(p);
    return cudaGetLastError();
}

}  // namespace mmbev
