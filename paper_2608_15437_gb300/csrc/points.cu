// Stage 1: the classify pass (S1 + S2 of the path).
//
// A persistent kernel, one block of 1,024 threads (32 warps) per SM,
// streams a contiguous range of 2,048-point tiles through a ring of 40 KB
// shared-memory buffers. Each tile arrives as eight 5 KB cp.async.bulk (TMA)
// copies with an L2 evict-first policy, counted on the buffer's mbarrier: on
// GB300 a single 40 KB bulk copy per tile streams at about a quarter of HBM
// bandwidth, eight concurrent ones at nearly all of it. The warps never wait
// for each other: they take 64-point chunks (32 to a tile) in increasing
// order from a shared-memory counter, each as soon as it has finished the
// last, and whichever warp finishes the last chunk of a buffer's tile (a
// shared-memory counter) refills it with the tile one ring length ahead. With
// a fixed chunk per warp and tile, warps instead polled the barrier of a tile
// that one slow chunk held back (chunks whose points meet many ROIs cost
// several times the others).
// Per point: Eq. 6 motion compensation, range crop, Alg. 1 inside-ROI test
// (coarse candidate mask, then the exact rotated-box test in rank order;
// the first hit is the point's rank; a point inside no ROI is kept with
// probability rho_out and rank R_f) and the voxel index. The masks and
// prepared ROIs of the (one or two) frames a block's tile range starts with
// sit in shared memory. Kept points are compacted per 32-point region with
// warp ballots, in input order: position (region)*32 + (rank among the
// region's kept points) gets a 32-byte record with the compensated features
// and the ROI rank, so later stages never touch the raw points again, and the
// point's frame and lin (frame << 32 | lin). Every region's kept count goes to a
// byte array, from which the compaction stage gathers the keys in position
// order.
//
// The classify-only entry point (per-point outputs for testing S1-S2) uses a
// plain one-thread-per-point kernel built from the same device functions.
#include <atomic>

#include "mmbev_internal.cuh"

namespace mmbev {
namespace {

constexpr int kThreads = 1024;
constexpr int kTileChunks = kTile / 64;       // 64-point chunks per tile (32)
constexpr int kTfStageMax = 512;              // sweeps whose transforms sit in smem
constexpr int kMaskSmemWords = 8192;          // largest staged coarse mask of a frame (32 KB)
constexpr int kChunks = 8;                    // bulk copies per tile
constexpr int kChunkBytes = kTileBytes / kChunks;
static_assert(kTile == kTileChunks * 2 * kRegion, "a chunk covers two regions of a tile");

// ---- TMA / mbarrier helpers (inline PTX)
__device__ __forceinline__ uint32_t smem_addr(const void* p) {
    return (uint32_t)__cvta_generic_to_shared(p);
}
__device__ __forceinline__ void mbar_init(uint64_t* bar, uint32_t count) {
    asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_addr(bar)), "r"(count)
                 : "memory");
}
__device__ __forceinline__ void mbar_fence_init() {
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
}
__device__ __forceinline__ void mbar_expect_tx(uint64_t* bar, uint32_t bytes) {
    asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(smem_addr(bar)),
                 "r"(bytes)
                 : "memory");
}
__device__ __forceinline__ bool mbar_try_wait(uint64_t* bar, uint32_t parity) {
    uint32_t ok;
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
        "selp.u32 %0, 1, 0, p;\n\t}"
        : "=r"(ok)
        : "r"(smem_addr(bar)), "r"(parity)
        : "memory");
    return ok != 0;
}
__device__ __forceinline__ uint64_t evict_last_policy() {
    uint64_t pol;
    asm volatile("createpolicy.fractional.L2::evict_last.b64 %0, 1.0;" : "=l"(pol));
    return pol;
}
__device__ __forceinline__ void st_u64_hint(unsigned long long* a, unsigned long long v, uint64_t pol) {
    asm volatile("st.global.L2::cache_hint.u64 [%0], %1, %2;" ::"l"(a), "l"(v), "l"(pol) : "memory");
}
__device__ __forceinline__ uint64_t evict_first_policy() {
    uint64_t pol;
    asm volatile("createpolicy.fractional.L2::evict_first.b64 %0, 1.0;" : "=l"(pol));
    return pol;
}
__device__ __forceinline__ void tma_load(void* dst, const void* src, uint32_t bytes,
                                         uint64_t* bar, uint64_t pol) {
    asm volatile(
        "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes.L2::cache_hint "
        "[%0], [%1], %2, [%3], %4;" ::"r"(smem_addr(dst)),
        "l"(src), "r"(bytes), "r"(smem_addr(bar)), "l"(pol)
        : "memory");
}

// Bounded wait on an mbarrier phase; false when the wait gave up.
__device__ __forceinline__ bool mbar_wait(uint64_t* bar, uint32_t parity) {
    for (uint32_t i = 0; i < kSpinLimit; ++i)
        if (mbar_try_wait(bar, parity)) return true;
    return false;
}

struct ClsSmem {
    float* stages;    // [nstages][kTile * 5]
    uint32_t* mask;   // [2][coarse^2 * mask_words] coarse masks of the staged frames
    RoiPrep* rois;    // [2][rmax] prepared ROIs of the staged frames
    float* tf;        // [S][12] when staged
    int64_t* soff;    // [S+1]
    int32_t* sfr;     // [S] frame of each sweep
    int32_t* sr0;     // [S] first ROI of that frame
    uint64_t* full;   // [nstages] tile arrived
    uint32_t* done;   // [nstages] warps finished with the buffer
    uint32_t* issued; // [nstages] fills issued into the buffer
    uint32_t* kept;   // [4] kept points of the block, -, next chunk, abort flag
};

__host__ __device__ inline size_t align16(size_t o) { return (o + 15) & ~(size_t)15; }

// g2w: words of one frame's coarse mask (coarse^2 * mask_words).
__host__ __device__ inline size_t classify_smem_bytes(int S, int rmax, int nstages, int g2w) {
    const bool tf_staged = S <= kTfStageMax;
    size_t o = (size_t)nstages * kTileBytes + 2 * (size_t)g2w * 4 + 2 * (size_t)rmax * 32;
    o += tf_staged ? (size_t)S * 48 : 0;
    o += (size_t)(S + 1) * 8 + (size_t)S * 8;
    o = align16(o);
    return o + (size_t)nstages * 8 + (size_t)nstages * 8 + 16;
}

__device__ __forceinline__ ClsSmem carve(unsigned char* smem, int S, int rmax, int g2w, bool tf_staged,
                                         int nstages) {
    ClsSmem s;
    size_t o = 0;
    s.stages = reinterpret_cast<float*>(smem);
    o += (size_t)nstages * kTileBytes;
    s.mask = reinterpret_cast<uint32_t*>(smem + o);
    o += 2 * (size_t)g2w * 4;
    s.rois = reinterpret_cast<RoiPrep*>(smem + o);
    o += 2 * (size_t)rmax * 32;
    s.tf = reinterpret_cast<float*>(smem + o);
    o += tf_staged ? (size_t)S * 48 : 0;
    s.soff = reinterpret_cast<int64_t*>(smem + o);
    o += (size_t)(S + 1) * 8;
    s.sfr = reinterpret_cast<int32_t*>(smem + o);
    o += (size_t)S * 4;
    s.sr0 = reinterpret_cast<int32_t*>(smem + o);
    o += (size_t)S * 4;
    o = align16(o);
    s.full = reinterpret_cast<uint64_t*>(smem + o);
    o += (size_t)nstages * 8;
    s.done = reinterpret_cast<uint32_t*>(smem + o);
    o += (size_t)nstages * 4;
    s.issued = reinterpret_cast<uint32_t*>(smem + o);
    o += (size_t)nstages * 4;
    s.kept = reinterpret_cast<uint32_t*>(smem + o);
    return s;
}

// Lanes 0..kChunks-1 of one warp each move one chunk of a tile into
// buffer `stage`.
__device__ __forceinline__ void issue_tile(const Params& p, const ClsSmem& sm, int stage,
                                           int64_t tile, int lane, uint64_t pol) {
    if (lane == 0) sm.issued[stage] += 1u;   // one warp refills a buffer at a time
    if (lane < kChunks) {
        const size_t off = (size_t)lane * kChunkBytes;
        mbar_expect_tx(&sm.full[stage], kChunkBytes);
        tma_load(reinterpret_cast<unsigned char*>(sm.stages + (size_t)stage * kTile * 5) + off,
                 reinterpret_cast<const unsigned char*>(p.points + tile * kTile * 5) + off,
                 kChunkBytes, &sm.full[stage], pol);
    }
}

// The block's tile range, chunk after chunk. Work is handed out in chunks of
// 64 points (a tile holds 32), in increasing order, from a shared-memory
// counter: a warp takes the next chunk as soon as it is done with its
// current one, so warps whose points meet many ROIs do not hold the others
// back. A buffer is refilled, with the tile one ring length ahead, by
// whichever warp finishes the last of its 32 chunks. Within a chunk, lane l
// takes points 2l and 2l+1: their ten floats are five 8-byte shared loads,
// conflict-free (lane stride 40 bytes). Lanes 0-15 cover the chunk's first
// 32-point region, lanes 16-31 its second. kStaged: every frame of the range
// has its mask and ROIs in shared memory. Point indices fit in 32 bits (the
// host rejects more points). Returns false when a wait gave up.
template <bool kStaged>
__device__ __forceinline__ bool classify_range(const Params& p, const ClsSmem& sm, int rmax,
                                               int nstages, int64_t t_begin, int64_t t_end,
                                               int f_lo, int n_staged) {
    const int lane = threadIdx.x & 31;
    const int S = p.num_sweeps;
    const bool tf_staged = S <= kTfStageMax;
    const uint32_t N = (uint32_t)p.num_points;
    const uint32_t full_tiles = N / kTile;
    const int G2W = p.coarse * p.coarse * p.mask_words;
    const uint64_t pol = evict_first_policy();
    const uint32_t lt = (1u << lane) - 1u;
    const uint32_t half_mask = lane < 16 ? 0x0000FFFFu : 0xFFFF0000u;
    const uint32_t nchunks = (uint32_t)(t_end - t_begin) * (uint32_t)kTileChunks;
    const uint32_t tb = (uint32_t)t_begin;
    // the sweep of this lane's current point and what depends on it (points
    // only move forward: chunks are taken in increasing order)
    int s = find_sweep(sm.soff, S, t_begin * kTile);
    uint32_t next_off = 0;     // first index of the next sweep
    float T[12];
    uint32_t fr = 0;
    uint32_t moff = 0, roff = 0;           // staged: the frame's mask / ROI offsets in shared memory
    const uint32_t* fmask = nullptr;       // not staged: its mask and ROIs in global memory
    const RoiPrep* frois = nullptr;
    auto load_sweep = [&]() {
        next_off = (uint32_t)sm.soff[s + 1];
        if (tf_staged) {
            const float4* t4 = reinterpret_cast<const float4*>(sm.tf + s * 12);
            const float4 a = t4[0], b = t4[1], c = t4[2];
            T[0] = a.x; T[1] = a.y; T[2] = a.z; T[3] = a.w;
            T[4] = b.x; T[5] = b.y; T[6] = b.z; T[7] = b.w;
            T[8] = c.x; T[9] = c.y; T[10] = c.z; T[11] = c.w;
        } else {
#pragma unroll
            for (int c = 0; c < 12; ++c) T[c] = __ldg(p.sweep_tf + (size_t)s * 16 + c);
        }
        const int f = sm.sfr[s];
        fr = (uint32_t)f;
        if (kStaged) {
            const int slot = f - f_lo;   // 0 or 1
            moff = (uint32_t)(slot * G2W);
            roff = (uint32_t)(slot * rmax);
        } else {
            const int slot = f - f_lo;
            if (slot >= 0 && slot < n_staged) {
                fmask = sm.mask + slot * G2W;
                frois = sm.rois + (size_t)slot * rmax;
            } else {
                fmask = p.masks + (size_t)f * G2W;
                frois = p.roi_prep + sm.sr0[s];
            }
        }
    };
    load_sweep();
    // ring position of tile t_begin + tt: buffer st, its round (fill count)
    uint32_t tt = 0, round = 0;
    int st = 0;
    uint32_t c = 0;
    if (lane == 0) c = atomicAdd(&sm.kept[2], 1u);
    c = __shfl_sync(0xFFFFFFFFu, c, 0);
    while (c < nchunks) {
        // another warp gave up waiting: stop taking chunks
        if (*reinterpret_cast<volatile uint32_t*>(&sm.kept[3])) return false;
        uint32_t cn = 0;   // the warp's next chunk, fetched early
        if (lane == 0) cn = atomicAdd(&sm.kept[2], 1u);
        const uint32_t ct = c / (uint32_t)kTileChunks, sub = c % (uint32_t)kTileChunks;
        while (tt < ct) {   // chunks only move forward
            ++tt;
            if (++st == nstages) {
                st = 0;
                ++round;
            }
        }
        const uint32_t tile = tb + ct;
        const uint32_t base = tile * (uint32_t)kTile;
        const uint32_t j0 = sub * 64u + 2u * (uint32_t)lane;
        const uint32_t i0 = base + j0;   // the lane's first point
        float2 v0, v1, v2, v3, v4;
        if (tile < full_tiles) {
            // A phase-parity wait only tells the phase it waits for from the
            // one before it. Chunks are handed out up to two per warp (64
            // chunks, two tiles) ahead of their buffers, and nothing orders
            // the arrival of tiles in flight: when later tiles land and are
            // done first, a warp can hold a chunk of a buffer's next round
            // before the current round's tile has landed, and would see the
            // previous round's phase as its own (with a ring of two buffers
            // that takes no reordering at all). So it first waits (bounded)
            // until every chunk of the buffer's previous round has released
            // it; the previous phase has completed by then.
            bool ok = true;
            if (round > 0u) {
                uint32_t spins = 0;
                while (*reinterpret_cast<volatile uint32_t*>(&sm.done[st]) <
                       round * (uint32_t)kTileChunks)
                    if (++spins >= kSpinLimit) {
                        ok = false;
                        break;
                    }
            }
            if (!ok || !mbar_wait(&sm.full[st], round & 1u)) {
                if (lane == 0) {
                    set_status(p.hdr, MMBEV_DEV_WAIT_TIMEOUT);
                    atomicExch(&sm.kept[3], 1u);
                }
                return false;
            }
            const float2* q2 =
                reinterpret_cast<const float2*>(sm.stages + (size_t)st * kTile * 5 + 5 * j0);
            v0 = q2[0]; v1 = q2[1]; v2 = q2[2]; v3 = q2[3]; v4 = q2[4];
        } else {
            // the ragged last tile never enters the ring: the lane reads its
            // points (those below N) from global memory
            const float* src = p.points + (size_t)i0 * 5;
            float q[10];
#pragma unroll
            for (int k = 0; k < 10; ++k) q[k] = i0 + k / 5 < N ? __ldcs(src + k) : 0.f;
            v0 = make_float2(q[0], q[1]); v1 = make_float2(q[2], q[3]);
            v2 = make_float2(q[4], q[5]); v3 = make_float2(q[6], q[7]);
            v4 = make_float2(q[8], q[9]);
        }
        // the chunk is done with the buffer once its reads are complete; the
        // last of the tile's 32 chunks refills it
        __threadfence_block();
        __syncwarp();
        {
            uint32_t last = 0;
            if (lane == 0)  // the counter only grows: a round ends at its kTileChunks-th arrival
                last = atomicAdd(&sm.done[st], 1u) == (round + 1u) * kTileChunks - 1u;
            last = __shfl_sync(0xFFFFFFFFu, last, 0);
            if (last) {
                const int64_t next = (int64_t)tile + nstages;
                if (next < t_end && next < (int64_t)full_tiles) issue_tile(p, sm, st, next, lane, pol);
            }
        }
        const float px[2] = {v0.x, v2.y}, py[2] = {v0.y, v3.x}, pz[2] = {v1.x, v3.y};
        const float pi[2] = {v1.y, v4.x}, pd[2] = {v2.x, v4.y};
        bool valid[2] = {false, false};
        uint32_t lin[2] = {0u, 0u}, frk[2] = {0u, 0u};
        int hit[2] = {-1, -1};
        float x[2], y[2], z[2];
        int cell[2] = {-1, -1};               // the point's coarse cell (-1: out of range)
        uint32_t cmo[2] = {0u, 0u}, cro[2] = {0u, 0u};
        const uint32_t* cm[2] = {nullptr, nullptr};
        const RoiPrep* cr[2] = {nullptr, nullptr};
        // a sweep boundary inside the chunk (rare) reloads per point
        const bool cross = __any_sync(0xFFFFFFFFu, i0 + 1u >= next_off);
#pragma unroll
        for (int k = 0; k < 2; ++k) {
            const uint32_t idx = i0 + (uint32_t)k;
            if (cross && idx >= next_off && idx < N) {
                while (s + 1 < S && (uint32_t)sm.soff[s + 1] <= idx) ++s;
                load_sweep();
            }
            compensate(T, px[k], py[k], pz[k], x[k], y[k], z[k]);
            int cl;
            if (idx < N && point_cell(p, x[k], y[k], z[k], cl)) cell[k] = cl;
            if (kStaged) {
                cmo[k] = moff;
                cro[k] = roff;
            } else {
                cm[k] = fmask;
                cr[k] = frois;
            }
            frk[k] = fr;
        }
        // Alg. 1 ROI test in rank order over the union of the warp's
        // candidates: each step tests one ROI index for all 64 points (a
        // broadcast read when the warp's points share a frame); a point keeps
        // its first hit.
        for (int w = 0; w < p.mask_words; ++w) {
            uint32_t m[2];
#pragma unroll
            for (int k = 0; k < 2; ++k) {
                m[k] = 0u;
                if (cell[k] >= 0 && hit[k] < 0) {
                    const int wi = cell[k] * p.mask_words + w;
                    m[k] = kStaged ? sm.mask[cmo[k] + wi] : cm[k][wi];
                }
            }
            uint32_t u = __reduce_or_sync(0xFFFFFFFFu, m[0] | m[1]);
            while (u) {
                const int b = __ffs(u) - 1;
                u &= u - 1u;
#pragma unroll
                for (int k = 0; k < 2; ++k)
                    if (((m[k] >> b) & 1u) && hit[k] < 0 &&
                        roi_hit(kStaged ? sm.rois + cro[k] : cr[k], w * 32 + b, x[k], y[k]))
                        hit[k] = w * 32 + b;
            }
        }
        // Alg. 1: an in-range point inside no ROI is kept with probability
        // rho_out (a SplitMix64 draw keyed by its index within the frame)
        if (p.rho_thr) {
#pragma unroll
            for (int k = 0; k < 2; ++k) {
                if (hit[k] >= 0 || cell[k] < 0) continue;
                const uint32_t f = frk[k];
                const int64_t j = (int64_t)(i0 + k) - sm.soff[p.frame_sweep_off[f]];
                if ((uint32_t)(splitmix64_nth(p.seed, (uint64_t)j + 1ull) >> 40) < p.rho_thr)
                    hit[k] = p.frame_roi_off[f + 1] - p.frame_roi_off[f];  // rank R_f
            }
        }
#pragma unroll
        for (int k = 0; k < 2; ++k) valid[k] = hit[k] >= 0 && voxel_lin(p, x[k], y[k], z[k], lin[k]);
        // compaction in the 32-point regions, input order kept: the record
        // position of a kept point grows with its index
        const uint32_t b0 = __ballot_sync(0xFFFFFFFFu, valid[0]);
        const uint32_t b1 = __ballot_sync(0xFFFFFFFFu, valid[1]);
        const uint32_t below = lt & half_mask;
        const uint32_t rank0 = __popc(b0 & below) + __popc(b1 & below);
        const uint32_t region = tile * (uint32_t)(kTile / kRegion) + sub * 2u + (uint32_t)(lane >> 4);
        // every region's kept count, so the compaction stage can find the
        // kept points' keys in position order
        if ((lane & 15) == 0)
            p.rcnt[region] = (uint8_t)(__popc(b0 & half_mask) + __popc(b1 & half_mask));
        const uint32_t nk = __popc(b0) + __popc(b1);
        if (nk == 0u) {   // warp-uniform: nothing kept in the chunk
            c = __shfl_sync(0xFFFFFFFFu, cn, 0);
            continue;
        }
        if (lane == 0) atomicAdd(&sm.kept[0], nk);
#pragma unroll
        for (int k = 0; k < 2; ++k) {
            if (valid[k]) {
                const uint32_t rk = rank0 + (k ? (uint32_t)valid[0] : 0u);
                const uint32_t at = region * (uint32_t)kRegion + rk;
                // records are read again only by the output stage: streaming
                // stores leave L2 to the keys in between
                uint4* rec = p.records + 2 * (size_t)at;
                __stcs(rec, make_uint4(__float_as_uint(x[k]), __float_as_uint(y[k]),
                                       __float_as_uint(z[k]), __float_as_uint(pi[k])));
                __stcs(rec + 1, make_uint4(__float_as_uint(pd[k]), (uint32_t)hit[k], 0u, 0u));
                // the sort key: the frame, the voxel's lin; kept in L2 past
                // the input stream for the compaction stage that reads it next
                st_u64_hint(p.ckey + at, (unsigned long long)frk[k] << 32 | lin[k],
                            evict_last_policy());
            }
        }
        c = __shfl_sync(0xFFFFFFFFu, cn, 0);
    }
    return true;
}

__global__ void __launch_bounds__(kThreads, 1) k_classify(Params p, int rmax, int nstages) {
    extern __shared__ __align__(128) unsigned char smem[];
    pdl_wait();
    const int t = threadIdx.x, lane = t & 31, warp = t >> 5;
    const int S = p.num_sweeps;
    const bool tf_staged = S <= kTfStageMax;
    const int G2W = p.coarse * p.coarse * p.mask_words;
    ClsSmem sm = carve(smem, S, rmax, G2W, tf_staged, nstages);

    const int64_t N = p.num_points;
    const int64_t num_tiles = (N + kTile - 1) / kTile;
    const int64_t full_tiles = N / kTile;
    const int64_t t_begin = (int64_t)blockIdx.x * num_tiles / gridDim.x;
    const int64_t t_end = ((int64_t)blockIdx.x + 1) * num_tiles / gridDim.x;
    if (t_begin >= t_end) return;

    for (int i = t; i <= S; i += kThreads) sm.soff[i] = p.sweep_off[i];
    for (int i = t; i < S; i += kThreads) {
        const int f = p.sweep_frame[i];
        sm.sfr[i] = f;
        sm.sr0[i] = p.frame_roi_off[f];
    }
    if (tf_staged)
        for (int i = t; i < S * 12; i += kThreads)
            sm.tf[i] = __ldg(p.sweep_tf + (size_t)(i / 12) * 16 + (i % 12));
    // the frame of the range's first point and the next one
    const int f_lo = p.sweep_frame[find_sweep(p.sweep_off, S, t_begin * kTile)];
    const int n_staged = f_lo + 1 < p.num_frames ? 2 : 1;
    for (int k = 0; k < n_staged; ++k) {
        const int f = f_lo + k;
        const int r0 = p.frame_roi_off[f];
        const int rn = min(p.frame_roi_off[f + 1] - r0, rmax);
        const uint32_t* gm = p.masks + (size_t)f * G2W;
        for (int i = t; i < G2W; i += kThreads) sm.mask[k * G2W + i] = gm[i];
        for (int i = t; i < rn * 2; i += kThreads)
            reinterpret_cast<float4*>(sm.rois + (size_t)k * rmax)[i] =
                reinterpret_cast<const float4*>(p.roi_prep + r0)[i];
    }
    const uint64_t pol = evict_first_policy();
    if (t == 0) {
        for (int s = 0; s < nstages; ++s) {
            mbar_init(&sm.full[s], kChunks);
            sm.done[s] = 0u;
            sm.issued[s] = 0u;
        }
        sm.kept[0] = sm.kept[1] = sm.kept[2] = sm.kept[3] = 0u;
        mbar_fence_init();
    }
    __syncthreads();
    if (warp == 0)
        for (int s = 0; s < nstages; ++s) {
            const int64_t tile = t_begin + s;
            if (tile < t_end && tile < full_tiles) issue_tile(p, sm, s, tile, lane, pol);
        }

    // The frames of the block's range: when the (at most two) staged ones
    // cover it, every mask and ROI read is a shared-memory read.
    const int64_t last_pt = (t_end * kTile < N ? t_end * kTile : N) - 1;
    const int f_hi = p.sweep_frame[find_sweep(p.sweep_off, S, last_pt)];
    if (f_hi - f_lo < n_staged)
        classify_range<true>(p, sm, rmax, nstages, t_begin, t_end, f_lo, n_staged);
    else
        classify_range<false>(p, sm, rmax, nstages, t_begin, t_end, f_lo, n_staged);
    __syncthreads();
    if (t != 0) return;
    if (sm.kept[3]) {
        // A wait gave up (the status word says so). Before the block exits,
        // every bulk copy still in flight into its shared memory must land:
        // a buffer has at most one fill outstanding, the last one issued, so
        // wait (bounded again) for that fill's phase. The block's list is
        // published as empty.
        for (int s = 0; s < nstages; ++s) {
            const uint32_t k = sm.issued[s];
            if (k > 0) (void)mbar_wait(&sm.full[s], (k - 1u) & 1u);
        }
        p.cls_cnt[blockIdx.x] = 0u;
        p.cls_flo[blockIdx.x] = (uint32_t)f_lo;
        return;
    }
    const uint32_t tot = sm.kept[0];
    p.cls_cnt[blockIdx.x] = tot;
    p.cls_flo[blockIdx.x] = (uint32_t)f_lo;
    if (tot) atomicAdd(&p.hdr->num_rec, tot);
}

// One thread per point: the per-point view of S1-S2 for testing.
__global__ void __launch_bounds__(256) k_classify_points(Params p) {
    pdl_wait();
    const int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    if (i >= p.num_points) return;
    const int s = find_sweep(p.sweep_off, p.num_sweeps, i);
    float T[12];
#pragma unroll
    for (int c = 0; c < 12; ++c) T[c] = __ldg(p.sweep_tf + (size_t)s * 16 + c);
    const float* q = p.points + i * 5;
    float x, y, z;
    compensate(T, __ldg(q), __ldg(q + 1), __ldg(q + 2), x, y, z);
    p.cls_xyz[i * 3 + 0] = x;
    p.cls_xyz[i * 3 + 1] = y;
    p.cls_xyz[i * 3 + 2] = z;
    const int f = p.sweep_frame[s];
    uint32_t lin = 0, r = 0;
    const bool kept = classify_point(
        p, p.masks + (size_t)f * p.coarse * p.coarse * p.mask_words,
        p.roi_prep + p.frame_roi_off[f], x, y, z, lin, r);
    p.cls_lin[i] = kept ? (int64_t)lin : (int64_t)-1;
    p.cls_rank[i] = kept ? (int32_t)r : -1;
}

}  // namespace

cudaError_t launch_classify(const Params& p, int rmax, int num_sms, bool pdl, cudaStream_t st) {
    if (p.num_points <= 0) return cudaSuccess;
    if (p.coarse * p.coarse * p.mask_words > kMaskSmemWords) return cudaErrorInvalidValue;
    if (rmax < 1) rmax = 1;
    constexpr size_t kSmemLimit = 227 * 1024;
    int nstages = 4;
    const int g2w = p.coarse * p.coarse * p.mask_words;
    while (nstages > 2 && classify_smem_bytes(p.num_sweeps, rmax, nstages, g2w) > kSmemLimit)
        --nstages;
    const size_t smem = classify_smem_bytes(p.num_sweeps, rmax, nstages, g2w);
    if (smem > kSmemLimit) return cudaErrorInvalidValue;
    static std::atomic<int> configured[64];
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    if (dev < 0 || dev >= 64 || !configured[dev].load(std::memory_order_acquire)) {
        e = cudaFuncSetAttribute(k_classify, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                 (int)kSmemLimit);
        if (e != cudaSuccess) return e;
        if (dev >= 0 && dev < 64) configured[dev].store(1, std::memory_order_release);
    }
    (void)num_sms;
    return launch_k(k_classify, dim3(p.cls_grid), dim3(kThreads), smem, st, pdl, p, rmax,
                    nstages);
}

cudaError_t launch_classify_points(const Params& p, cudaStream_t st) {
    if (p.num_points <= 0) return cudaSuccess;
    const int64_t blocks = (p.num_points + 255) / 256;
    return launch_k(k_classify_points, dim3((unsigned)blocks), dim3(256), 0, st, false, p);
}

}  // namespace mmbev
