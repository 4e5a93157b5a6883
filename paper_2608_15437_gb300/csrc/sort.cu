// Stages 2-5: voxel dedup (S3), cap and canonical order (S4), first-K mean
// features (S5) of the path (Alg. 1 "Voxelize" and "VoxelFeatureEncoder";
// Sec. IV-F hard voxelization; Sec. IV-C mandatory ROIs first).
//
// Every kept point has a 32-byte record at its position (positions ascend
// with the point index) and its frame and lin. The stages sort each frame's
// kept points by lin with a stable least-significant-digit radix sort,
// starting from position order, so that each voxel's points end up as one
// run, runs in ascending lin, and a run's points in ascending position: a
// voxel's first K points by index are the first K of its run. Frames are
// independent problems and every chain of tiles below stays within one
// frame, so a tile's look-back never walks further than its frame's start.
//
//   compact  (stage 2)  the kept points' lins and positions in position
//                       order, hence frame after frame (a scan of the
//                       regions' kept counts, chained across tiles by
//                       decoupled look-back), each frame's kept count, and
//                       the histogram of each frame's lin digits.
//   sort     (stage 3)  one launch per 9-bit digit, lowest first; tiles of
//                       4,096 items within a frame: items take their rank
//                       among the tile's items of their digit in item order
//                       (warp match on the digit, a count per warp and
//                       digit), the digit's offset in the frame comes from
//                       the frame's histogram and a decoupled look-back over
//                       the frame's earlier tiles, and the item moves there.
//                       Stable, so the passes compose.
//   runs     (stage 4)  a run starts where the lin changes: run heads are
//                       numbered within each frame (a scan chained by
//                       look-back over the frame's tiles); voxel v of frame f
//                       gets its run's first and end items and its lin, and
//                       the frame's last tile its voxel count.
//   emit     (stage 5)  a thread per output row: a frame within max_voxels
//                       keeps every voxel, row = its index in the frame; the
//                       fp32 sum of the first K records of the run in order,
//                       one IEEE divide, coordinates, count. A frame over
//                       the cap (a block) keeps the max_voxels smallest by
//                       (minimum rank, lin): minimum ranks of its voxels from
//                       their records, their histogram gives the threshold
//                       rank r* and the quota q of rank-r* voxels, which are
//                       kept in ascending lin.
#include <atomic>

#include "mmbev_internal.cuh"

namespace mmbev {
namespace {

constexpr uint32_t kFull = 0xFFFFFFFFu;
// Look-back words: the value in the low 32 bits, a flag above.
constexpr unsigned long long kAgg = 1ull << 32;    // the tile's own total published
constexpr unsigned long long kInc = 2ull << 32;    // its inclusive prefix published
constexpr unsigned long long kFlags = 3ull << 32;

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

// Bounded wait for a published look-back word (relaxed loads: the word is
// its own payload); after the first few polls the thread backs off, so that
// many waiting threads do not crowd L2. False when the wait gave up.
__device__ __forceinline__ bool poll_word(const unsigned long long* a, unsigned long long& w) {
    for (uint32_t i = 0; i < kSpinLimit; ++i) {
        w = ld_relaxed(a);
        if (w & kFlags) return true;
        if (i >= 8) __nanosleep(64);
    }
    return false;
}

// Decoupled look-back by one warp over a chain of tiles `first` .. `tile`
// whose words are `st`: the tile publishes its total, then sums the totals of
// the tiles before it (32 at a time, each lane waiting, bounded, for its
// tile's word) until one carries an inclusive prefix (a tile before `first`
// counts as an inclusive 0), and publishes its own. Tiles are numbered in the
// order their blocks took them, so a tile only ever waits on tiles whose
// blocks are running. Returns the tile's exclusive prefix within the chain (in
// every lane); a wait that gives up sets the status and leaves the results
// void.
__device__ uint32_t lookback(unsigned long long* st, uint32_t tile, uint32_t first,
                             uint32_t total, Header* hdr) {
    const int lane = threadIdx.x & 31;
    if (tile == first) {
        if (lane == 0) atomicExch(&st[tile], kInc | total);
        return 0u;
    }
    if (lane == 0) atomicExch(&st[tile], kAgg | total);
    uint32_t base = 0;
    int64_t j = (int64_t)tile - 1;
    for (;;) {
        const int64_t q = j - lane;
        unsigned long long w = kInc;   // before the chain: an inclusive prefix of 0
        bool gave_up = false;
        if (q >= (int64_t)first) gave_up = !poll_word(&st[q], w);
        if (__any_sync(kFull, gave_up)) {
            if (lane == 0) set_status(hdr, MMBEV_DEV_WAIT_TIMEOUT);
            break;
        }
        const uint32_t inc = __ballot_sync(kFull, (w & kInc) != 0ull);
        const int last = inc ? __ffs(inc) - 1 : 31;   // lanes 0..last contribute
        uint32_t v = lane <= last ? (uint32_t)w : 0u;
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(kFull, v, o);
        base += v;
        if (inc) break;
        j -= 32;
    }
    if (lane == 0) atomicExch(&st[tile], kInc | (unsigned long long)(base + total));
    return base;
}

// Per frame, exclusive prefixes of the kept counts (its first item,
// s_fstart) and of the tiles of `tile` items its items take (s_tpre); F + 1
// entries each. Every thread must call it.
template <int NT>
__device__ __forceinline__ void frame_tables(const Params& p, uint32_t tile, uint32_t* s_fstart,
                                             uint32_t* s_tpre, uint32_t* s_warp) {
    constexpr int per = (kMaxFrames + NT - 1) / NT;
    const int t = threadIdx.x;
    const uint32_t F = (uint32_t)p.num_frames;
    uint32_t c[per], n[per], sc = 0, sn = 0;
#pragma unroll
    for (int k = 0; k < per; ++k) {
        const uint32_t f = (uint32_t)t * per + k;
        c[k] = f < F ? p.fcnt[f] : 0u;
        n[k] = (c[k] + tile - 1u) / tile;
        sc += c[k];
        sn += n[k];
    }
    uint32_t tc = 0, tn = 0;
    uint32_t ec = block_exclusive_scan(sc, s_warp, &tc);
    uint32_t en = block_exclusive_scan(sn, s_warp, &tn);
#pragma unroll
    for (int k = 0; k < per; ++k) {
        const uint32_t f = (uint32_t)t * per + k;
        if (f < F) {
            s_fstart[f] = ec;
            if (s_tpre) s_tpre[f] = en;
        }
        ec += c[k];
        en += n[k];
    }
    if (t == 0) {
        s_fstart[F] = tc;
        if (s_tpre) s_tpre[F] = tn;
    }
    __syncthreads();
}

// The frame of tile `tile`: the largest f with s_tpre[f] <= tile (frames
// with no items take no tiles).
__device__ __forceinline__ uint32_t tile_frame(const uint32_t* s_tpre, uint32_t F, uint32_t tile) {
    uint32_t lo = 0, hi = F;   // s_tpre[lo] <= tile < s_tpre[hi]
    while (hi - lo > 1) {
        const uint32_t mid = (lo + hi) >> 1;
        if (s_tpre[mid] <= tile) lo = mid; else hi = mid;
    }
    return lo;
}

// ------------------------------------------------------------------ stage 2

constexpr int kCT = 1024;                      // threads of a compaction block
constexpr int kCW = kCT / 32;
constexpr uint32_t kCRound = 2 * kCT;          // regions a round (two a thread)
constexpr int kCU = 4;                         // entries a thread moves at once
// dynamic shared memory: a round's entry -> region table (two bytes an
// entry), its regions' first entries, the range's first two frames' digit
// histograms
constexpr size_t kCTabBytes = (size_t)kCRound * kRegion * 2;
constexpr size_t kCSmem = kCTabBytes + (size_t)kCRound * 4 + 2 * (size_t)kMaxPasses * kDigits * 4;

// A block per classify block: it takes the same range of point tiles, whose
// kept points are the ones after those of the classify blocks before it
// (their kept counts), so no block waits for another. In rounds of kCRound
// regions, a thread holds two regions' kept counts; a block scan gives each
// region its first entry, and a table in shared memory the region of every
// entry of the round. Thread t then moves entries t, t + kCT, ... (lin and
// position, into buffer A at the range's first index + the entry), counting
// each into its frame's kept count and digit histograms (shared memory for
// the range's first two frames, which are all its frames unless frames are
// small; others straight to global memory), added to the frames' totals at
// the end.
__global__ void __launch_bounds__(kCT) k_compact(Params p) {
    extern __shared__ __align__(16) unsigned char c_smem[];
    uint16_t* s_tab = reinterpret_cast<uint16_t*>(c_smem);
    uint32_t* s_rpre = reinterpret_cast<uint32_t*>(c_smem + kCTabBytes);
    uint32_t* s_h = s_rpre + kCRound;   // [2][kMaxPasses * kDigits]
    __shared__ uint32_t s_warp[kCW];
    __shared__ uint32_t s_fc[2];
    __shared__ uint32_t s_base;
    pdl_wait();
    const int t = threadIdx.x, lane = t & 31;
    const uint32_t M = p.hdr->num_rec;
    const uint32_t F = (uint32_t)p.num_frames;
    const int P = p.sort_passes;
    {
        // the look-back words of the first radix pass and of the voxel
        // numbering start at zero (for as many tiles as M items can take)
        const size_t gt = (size_t)blockIdx.x * kCT + t, gs = (size_t)gridDim.x * kCT;
        const size_t st = min((size_t)(M + kSortTile - 1) / kSortTile + F, (size_t)p.sort_tiles_cap);
        for (size_t i = gt; i < st * kDigits; i += gs) p.sort_state[i] = 0ull;
        const size_t rt = min((size_t)(M + kRunTile - 1) / kRunTile + F, (size_t)p.run_tiles_cap);
        for (size_t i = gt; i < rt; i += gs) p.run_state[i] = 0ull;
    }
    for (int i = t; i < 2 * kMaxPasses * kDigits; i += kCT) s_h[i] = 0u;
    if (t < 2) s_fc[t] = 0u;
    {
        // kept points of the classify blocks before this one
        const uint32_t x = (uint32_t)t < blockIdx.x && t < kMaxClsGrid ? p.cls_cnt[t] : 0u;
        uint32_t tot = 0;
        (void)block_exclusive_scan(x, s_warp, &tot);
        if (t == 0) s_base = tot;
    }
    // the classify block's range of point tiles, split as the classify kernel
    // splits it, and the frame of its first point
    const uint64_t num_tiles = ((uint64_t)p.num_points + kTile - 1) / kTile;
    const uint64_t t0 = (uint64_t)blockIdx.x * num_tiles / gridDim.x;
    const uint64_t t1 = ((uint64_t)blockIdx.x + 1) * num_tiles / gridDim.x;
    const uint32_t r0 = (uint32_t)t0 * (kTile / kRegion), r1 = (uint32_t)t1 * (kTile / kRegion);
    const uint32_t f_lo = p.cls_flo[blockIdx.x];
    __syncthreads();
    uint32_t carry = s_base;
    for (uint32_t rb = r0; rb < r1; rb += kCRound) {   // block-uniform
        const uint32_t ra = rb + 2u * (uint32_t)t;
        uint32_t c0 = 0u, c1 = 0u;
        if (ra < r1) {   // r0 and r1 are even: two counts in one 16-bit word
            const uint32_t w2 = reinterpret_cast<const uint16_t*>(p.rcnt)[ra >> 1];
            c0 = min(w2 & 0xFFu, (uint32_t)kRegion);
            c1 = min(w2 >> 8, (uint32_t)kRegion);
        }
        uint32_t tot = 0;
        const uint32_t excl = block_exclusive_scan(c0 + c1, s_warp, &tot);
        s_rpre[2 * t] = excl;
        s_rpre[2 * t + 1] = excl + c0;
        for (uint32_t j = 0; j < c0; ++j) s_tab[excl + j] = (uint16_t)(2 * t);
        for (uint32_t j = 0; j < c1; ++j) s_tab[excl + c0 + j] = (uint16_t)(2 * t + 1);
        __syncthreads();
        for (uint32_t e0 = 0; e0 < tot; e0 += kCU * kCT) {   // block-uniform
            // kCU entries a thread, their loads issued before any is used
            uint32_t pos[kCU];
            unsigned long long key[kCU];
#pragma unroll
            for (int u = 0; u < kCU; ++u) {
                const uint32_t e = e0 + (uint32_t)u * kCT + (uint32_t)t;
                const uint32_t r = e < tot ? s_tab[e] : 0u;
                pos[u] = (rb + r) * (uint32_t)kRegion + (e - s_rpre[r]);
                key[u] = e < tot && pos[u] < p.rec_cap ? p.ckey[pos[u]] : ~0ull;
            }
#pragma unroll
            for (int u = 0; u < kCU; ++u) {
                const uint32_t e = e0 + (uint32_t)u * kCT + (uint32_t)t;
                const bool in = e < tot;
                const uint32_t f = (uint32_t)(key[u] >> 32), lin = (uint32_t)key[u];
                const uint32_t d = carry + e;
                const bool ok = in && pos[u] < p.rec_cap && f < F && d < p.rec_cap;
                if (in && !ok) set_status(p.hdr, MMBEV_DEV_BOUNDS);
                if (ok) {
                    p.key_a[d] = lin;
                    p.val_a[d] = pos[u];
                }
                // the frame's kept count and its digit histograms
                const uint32_t slot = f - f_lo;
                const uint32_t b0 = __ballot_sync(kFull, ok && slot == 0u);
                const uint32_t b1 = __ballot_sync(kFull, ok && slot == 1u);
                if (lane == 0) {
                    if (b0) atomicAdd(&s_fc[0], (uint32_t)__popc(b0));
                    if (b1) atomicAdd(&s_fc[1], (uint32_t)__popc(b1));
                }
                if (ok && slot > 1u) atomicAdd(&p.fcnt[f], 1u);
                if (ok) {
                    for (int q = 0; q < P; ++q) {
                        const uint32_t dg = (lin >> (kDigitBits * q)) & (kDigits - 1u);
                        if (slot <= 1u) atomicAdd(&s_h[slot * kMaxPasses * kDigits + q * kDigits + dg], 1u);
                        else atomicAdd(&p.hist[((size_t)f * kMaxPasses + q) * kDigits + dg], 1u);
                    }
                }
            }
        }
        carry += tot;
        __syncthreads();   // the table is rewritten by the next round
    }
    for (uint32_t slot = 0; slot < 2u; ++slot) {
        const uint32_t f = f_lo + slot;
        if (f >= F) break;
        const uint32_t* h = s_h + slot * kMaxPasses * kDigits;
        for (int i = t; i < P * kDigits; i += kCT)
            if (h[i]) atomicAdd(&p.hist[(size_t)f * kMaxPasses * kDigits + i], h[i]);
        if (t == 0 && s_fc[slot]) atomicAdd(&p.fcnt[f], s_fc[slot]);
    }
}

// ------------------------------------------------------------------ stage 3

constexpr int kST = 512;                       // threads of a radix pass block
constexpr int kSW = kST / 32;                  // 16 warps
constexpr int kSI = kSortTile / kST;           // 8 items a thread
static_assert(kSI * kST == (int)kSortTile, "tile");
static_assert(kST == kDigits, "a thread per digit in the look-back");

// One LSD pass over digit `pass` (bits 9*pass .. 9*pass+8) of the lins,
// within each frame. A frame's items are cut into tiles from its first item;
// items of a tile are taken warp by warp, 256 a warp in 8 rounds of 32,
// which is their order. Persistent blocks take tiles in order (frame by
// frame).
__global__ void __launch_bounds__(kST, 2)
k_sort_pass(Params p, int pass, const uint32_t* __restrict__ kin, const uint32_t* __restrict__ vin,
            uint32_t* __restrict__ kout, uint32_t* __restrict__ vout) {
    __shared__ uint32_t s_wh[kSW][kDigits];   // per warp and digit: count, then the warp's offset
    __shared__ uint32_t s_fdoff[kDigits];     // the digit's first index within the frame
    __shared__ uint32_t s_goff[kDigits];      // ... plus the frame's first item and earlier tiles'
    __shared__ uint32_t s_fstart[kMaxFrames + 1];
    __shared__ uint32_t s_tpre[kMaxFrames + 1];
    __shared__ uint32_t s_warp[kSW];
    __shared__ uint32_t s_tile;
    pdl_wait();
    const int t = threadIdx.x, lane = t & 31, warp = t >> 5;
    const uint32_t F = (uint32_t)p.num_frames;
    frame_tables<kST>(p, kSortTile, s_fstart, s_tpre, s_warp);
    const uint32_t T = min(s_tpre[F], p.sort_tiles_cap);
    const size_t slab = (size_t)p.sort_tiles_cap * kDigits;
    unsigned long long* st = p.sort_state + (size_t)(pass & 1) * slab;
    {
        // the next pass's look-back words start at zero (the previous pass,
        // which used them, is complete)
        unsigned long long* nx = p.sort_state + (size_t)((pass + 1) & 1) * slab;
        const size_t gt = (size_t)blockIdx.x * kST + t, gs = (size_t)gridDim.x * kST;
        for (size_t i = gt; i < (size_t)T * kDigits; i += gs) nx[i] = 0ull;
    }
    const int shift = kDigitBits * pass;
    const uint32_t lt = (1u << lane) - 1u;
    uint32_t cur_f = kUnset;   // the frame whose digit offsets s_fdoff holds
    for (;;) {
        if (t == 0) s_tile = atomicAdd(&p.hdr->sort_ticket[pass], 1u);
        for (int i = t; i < kSW * kDigits; i += kST) (&s_wh[0][0])[i] = 0u;
        __syncthreads();
        const uint32_t tile = s_tile;
        if (tile >= T) break;
        const uint32_t f = tile_frame(s_tpre, F, tile);
        const uint32_t ft = tile - s_tpre[f];   // the tile's place in its frame
        if (f != cur_f) {   // block-uniform
            const uint32_t h = p.hist[((size_t)f * kMaxPasses + pass) * kDigits + t];
            uint32_t tot = 0;
            s_fdoff[t] = block_exclusive_scan(h, s_warp, &tot);
            cur_f = f;
        }
        const uint32_t fend = s_fstart[f + 1];
        const uint32_t base =
            s_fstart[f] + ft * kSortTile + (uint32_t)warp * (32u * kSI) + (uint32_t)lane;
        uint32_t k[kSI], v[kSI], d[kSI], r[kSI];
#pragma unroll
        for (int j = 0; j < kSI; ++j) {
            const uint32_t idx = base + 32u * j;
            const bool ok = idx < fend;
            k[j] = ok ? kin[idx] : kNoLin;
            v[j] = ok ? vin[idx] : 0u;
            d[j] = ok ? (k[j] >> shift) & (kDigits - 1u) : (uint32_t)kDigits;
        }
        // rank among the warp's items of the same digit, in item order
#pragma unroll
        for (int j = 0; j < kSI; ++j) {
            const uint32_t peers = __match_any_sync(kFull, d[j]);
            const uint32_t before = __popc(peers & lt);
            const uint32_t old = d[j] < (uint32_t)kDigits ? s_wh[warp][d[j]] : 0u;
            __syncwarp();
            if (d[j] < (uint32_t)kDigits && before == 0u) s_wh[warp][d[j]] = old + __popc(peers);
            __syncwarp();
            r[j] = old + before;
        }
        __syncthreads();
        {
            // digit t: the warps' offsets within the tile, the tile's count
            uint32_t run = 0;
#pragma unroll
            for (int w = 0; w < kSW; ++w) {
                const uint32_t x = s_wh[w][t];
                s_wh[w][t] = run;
                run += x;
            }
            // decoupled look-back for digit t over the frame's earlier tiles
            unsigned long long* sw = st + (size_t)tile * kDigits + t;
            uint32_t excl = 0;
            if (ft == 0u) {
                atomicExch(sw, kInc | run);
            } else {
                atomicExch(sw, kAgg | run);
                // four of the earlier tiles' words at a time; a word not yet
                // published is waited for (bounded) before it is summed
                const uint32_t first = tile - ft;
                bool done = false;
                for (uint32_t q = tile - 1u; !done; q -= 4u) {
                    unsigned long long w[4];
#pragma unroll
                    for (int i = 0; i < 4; ++i)
                        w[i] = q >= first + (uint32_t)i ? ld_relaxed(st + (size_t)(q - i) * kDigits + t)
                                                        : kInc;
#pragma unroll
                    for (int i = 0; i < 4; ++i) {
                        if (done) break;
                        if ((w[i] & kFlags) == 0ull &&
                            !poll_word(st + (size_t)(q - i) * kDigits + t, w[i])) {
                            set_status(p.hdr, MMBEV_DEV_WAIT_TIMEOUT);
                            done = true;
                            break;
                        }
                        excl += (uint32_t)w[i];
                        if (w[i] & kInc) done = true;
                    }
                }
                atomicExch(sw, kInc | (unsigned long long)(excl + run));
            }
            s_goff[t] = s_fstart[f] + s_fdoff[t] + excl;
        }
        __syncthreads();
#pragma unroll
        for (int j = 0; j < kSI; ++j) {
            if (d[j] < (uint32_t)kDigits) {
                const uint32_t dst = s_goff[d[j]] + s_wh[warp][d[j]] + r[j];
                if (dst < fend) {
                    kout[dst] = k[j];
                    vout[dst] = v[j];
                } else {
                    set_status(p.hdr, MMBEV_DEV_BOUNDS);
                }
            }
        }
        __syncthreads();   // s_wh, s_goff and s_tile are rewritten for the next tile
    }
}

// ------------------------------------------------------------------ stage 4

constexpr int kRT = 256;                       // threads of a numbering block
constexpr int kRI = kRunTile / kRT;            // 8 consecutive items a thread
static_assert(kRI * kRT == (int)kRunTile, "tile");

// Heads (first item of a run) and tails (last item) of each frame's sorted
// lins. Voxel v of frame f, the v-th head of the frame, gets {head item,
// tail item + 1, lin} at vdesc[(frame's first item) + v] (the head writes
// words x, z, w and the tail word y); the frame's last tile writes its
// voxel count.
__global__ void __launch_bounds__(kRT) k_runs(Params p) {
    __shared__ uint32_t s_fstart[kMaxFrames + 1];
    __shared__ uint32_t s_tpre[kMaxFrames + 1];
    __shared__ uint32_t s_warp[kRT / 32];
    __shared__ uint32_t s_tile, s_base;
    pdl_wait();
    const int t = threadIdx.x;
    const uint32_t F = (uint32_t)p.num_frames;
    const uint32_t* K = p.skey;
    frame_tables<kRT>(p, kRunTile, s_fstart, s_tpre, s_warp);
    const uint32_t T = min(s_tpre[F], p.run_tiles_cap);
    uint32_t* vd = reinterpret_cast<uint32_t*>(p.vdesc);
    for (;;) {
        __syncthreads();
        if (t == 0) s_tile = atomicAdd(&p.hdr->run_ticket, 1u);
        __syncthreads();
        const uint32_t tile = s_tile;
        if (tile >= T) break;
        const uint32_t f = tile_frame(s_tpre, F, tile);
        const uint32_t ft = tile - s_tpre[f];
        const uint32_t fbeg = s_fstart[f], fend = s_fstart[f + 1];
        const uint32_t i0 = fbeg + ft * kRunTile + (uint32_t)t * kRI;
        uint32_t key[kRI + 2];   // items i0-1 .. i0+kRI (kNoLin outside the frame)
        key[0] = i0 > fbeg && i0 <= fend ? K[i0 - 1u] : kNoLin;
#pragma unroll
        for (int j = 0; j <= kRI; ++j) key[j + 1] = i0 + j < fend ? K[i0 + j] : kNoLin;
        uint32_t heads = 0u;
#pragma unroll
        for (int j = 0; j < kRI; ++j)
            if (i0 + j < fend && key[j + 1] != key[j]) heads |= 1u << j;
        uint32_t tot = 0;
        const uint32_t excl = block_exclusive_scan(__popc(heads), s_warp, &tot);
        if (t < 32) {
            const uint32_t b = lookback(p.run_state, tile, tile - ft, tot, p.hdr);
            if (t == 0) {
                s_base = b;
                if (tile + 1u == s_tpre[f + 1]) p.ftot[f] = b + tot;   // the frame's last tile
            }
        }
        __syncthreads();
        uint32_t g = fbeg + s_base + excl;   // the voxel of the next head
#pragma unroll
        for (int j = 0; j < kRI; ++j) {
            const uint32_t i = i0 + j;
            if (i >= fend) break;
            if (heads >> j & 1u) {
                if (g < fend) {
                    vd[4 * (size_t)g + 0] = i;
                    vd[4 * (size_t)g + 2] = key[j + 1];
                    vd[4 * (size_t)g + 3] = kUnset;
                } else {
                    set_status(p.hdr, MMBEV_DEV_BOUNDS);
                }
                ++g;
            }
            if (key[j + 2] != key[j + 1] && g > fbeg && g - 1u < fend)   // a tail
                vd[4 * (size_t)(g - 1u) + 1] = i + 1u;
        }
    }
}

// ------------------------------------------------------------------ stage 5

constexpr int kOutThreads = 256;
constexpr uint32_t kChunkRows = kOutThreads;   // rows a chunk of the output stage

// record: {x', y', z', intensity} {dt, rank, -, -}
__device__ __forceinline__ void add_record(float (&acc)[5], const uint4& a, float dt) {
    acc[0] = __fadd_rn(acc[0], __uint_as_float(a.x));
    acc[1] = __fadd_rn(acc[1], __uint_as_float(a.y));
    acc[2] = __fadd_rn(acc[2], __uint_as_float(a.z));
    acc[3] = __fadd_rn(acc[3], __uint_as_float(a.w));
    acc[4] = __fadd_rn(acc[4], dt);
}

// Voxel at vdesc[g] (of frame f, items [fbeg, fend)) into output row `row`:
// the fp32 sum of the records of the first min(count, K) points of its run,
// in order (ascending position, i.e. ascending index), one divide, its count
// and its coordinates.
template <int B>
__device__ __forceinline__ void emit_voxel(const Params& p, uint32_t f, uint32_t row, uint32_t g,
                                           uint32_t fbeg, uint32_t fend) {
    const uint4 d = p.vdesc[g];
    if (!(fbeg <= d.x && d.x < d.y && d.y <= fend)) {
        set_status(p.hdr, MMBEV_DEV_BOUNDS);
        return;
    }
    const uint32_t kept = min(d.y - d.x, (uint32_t)p.K);
    uint32_t pos[B];
#pragma unroll
    for (int j = 0; j < B; ++j) pos[j] = (uint32_t)j < kept ? p.sval[d.x + j] : 0u;
    constexpr int R = B < 2 ? B : 2;   // record loads in flight
    float acc[5] = {0.f, 0.f, 0.f, 0.f, 0.f};
#pragma unroll
    for (int j0 = 0; j0 < B; j0 += R) {
        if ((uint32_t)j0 >= kept) break;
        uint4 ra[R];
        float dt[R];
#pragma unroll
        for (int c = 0; c < R; ++c)
            if ((uint32_t)(j0 + c) < kept) {
                const uint32_t q = pos[j0 + c];
                if (q >= p.rec_cap) set_status(p.hdr, MMBEV_DEV_BOUNDS);
                const uint4* rec = p.records + 2 * (size_t)min(q, p.rec_cap - 1u);
                ra[c] = __ldg(rec);
                dt[c] = __ldg(reinterpret_cast<const float*>(rec + 1));
            }
#pragma unroll
        for (int c = 0; c < R; ++c)
            if ((uint32_t)(j0 + c) < kept) add_record(acc, ra[c], dt[c]);
    }
    const size_t r = (size_t)f * (uint32_t)p.max_voxels + row;
    const float fc = (float)kept;
#pragma unroll
    for (int c = 0; c < 5; ++c) p.out_feats[r * 5 + c] = __fdiv_rn(acc[c], fc);
    const uint32_t lin = d.z;
    const uint32_t q = udiv(p.div_nx, lin);      // cz * ny + cy
    const uint32_t cz = udiv(p.div_ny, q);
    p.out_coords[r * 3 + 0] = (int32_t)cz;
    p.out_coords[r * 3 + 1] = (int32_t)(q - cz * p.dims[1]);
    p.out_coords[r * 3 + 2] = (int32_t)(lin - q * p.dims[0]);
    p.out_counts[r] = (int32_t)kept;
}

// A frame over the cap, by one block: every voxel's minimum ROI rank (over
// all its points, from their records), their histogram, the threshold rank
// r* and quota q, then every kept voxel's row in ascending lin: a voxel below
// r* takes (voxels below r* before it) + min(ties before it, q); a voxel at
// r* is kept when fewer than q ties precede it.
template <int B>
__device__ void capped_frame(const Params& p, uint32_t f, uint32_t fbeg, uint32_t fend,
                             uint32_t* s_hist, uint32_t* s_warp) {
    const int t = threadIdx.x, lane = t & 31, warp = t >> 5;
    constexpr int nwarps = kOutThreads / 32;
    const uint32_t U = p.ftot[f];
    const uint32_t rn = (uint32_t)(p.frame_roi_off[f + 1] - p.frame_roi_off[f]);   // background rank
    const uint32_t maxv = (uint32_t)p.max_voxels;
    __shared__ uint32_t s_rstar, s_q;
    for (uint32_t r = t; r <= rn; r += kOutThreads) s_hist[r] = 0u;
    __syncthreads();
    uint32_t* vd = reinterpret_cast<uint32_t*>(p.vdesc);
    for (uint32_t v = warp; v < U; v += nwarps) {
        const uint4 d = p.vdesc[fbeg + v];
        uint32_t m = kUnset;
        if (fbeg <= d.x && d.x < d.y && d.y <= fend) {
            for (uint32_t j = d.x + lane; j < d.y; j += 32) {
                const uint32_t q = p.sval[j];
                if (q < p.rec_cap)
                    m = min(m, reinterpret_cast<const uint32_t*>(p.records + 2 * (size_t)q + 1)[1]);
            }
        } else if (lane == 0) {
            set_status(p.hdr, MMBEV_DEV_BOUNDS);
        }
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) m = min(m, __shfl_xor_sync(kFull, m, o));
        m = min(m, rn);
        if (lane == 0) {
            vd[4 * (size_t)(fbeg + v) + 3] = m;
            atomicAdd(&s_hist[m], 1u);
        }
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
    uint32_t ca = 0, cc = 0;   // voxels below r* and at r* before this round
    for (uint32_t v0 = 0; v0 < U; v0 += kOutThreads) {
        const uint32_t v = v0 + (uint32_t)t;
        const uint32_t r = v < U ? p.vdesc[fbeg + v].w : kUnset;
        const uint32_t b = r < rstar, c = r == rstar;
        uint32_t tb = 0, tc = 0;
        const uint32_t eb = block_exclusive_scan(b, s_warp, &tb);
        const uint32_t ec = block_exclusive_scan(c, s_warp, &tc);
        const uint32_t ab = ca + eb, cb = cc + ec;
        uint32_t row = kUnset;
        if (b) row = ab + min(cb, q);
        else if (c && cb < q) row = ab + cb;
        if (row != kUnset) {
            if (row < maxv) emit_voxel<B>(p, f, row, fbeg + v, fbeg, fend);
            else set_status(p.hdr, MMBEV_DEV_BOUNDS);
        }
        ca += tb;
        cc += tc;
    }
}

// Persistent blocks. Each first takes frames over the cap (a block each),
// then chunks of kChunkRows output rows of the other frames.
template <int B>
__global__ void __launch_bounds__(kOutThreads, (B <= 12 ? 6 : 2)) k_emit(Params p) {
    __shared__ uint32_t s_warp[kOutThreads / 32];
    __shared__ uint32_t s_fstart[kMaxFrames + 1];
    __shared__ uint32_t s_cpre[kMaxFrames + 1];   // chunks before each frame
    __shared__ uint32_t s_hist[kMaxRoisPerFrame + 2];
    __shared__ int s_bad;
    pdl_wait();
    const int t = threadIdx.x;
    const uint32_t F = (uint32_t)p.num_frames;
    const uint32_t maxv = (uint32_t)p.max_voxels;
    frame_tables<kOutThreads>(p, 1u, s_fstart, nullptr, s_warp);
    // the frames' items end within the kept points and their voxels within
    // their items, or nothing is written (a wait of an earlier stage gave up)
    if (t == 0) s_bad = s_fstart[F] != p.hdr->num_rec || s_fstart[F] > p.rec_cap;
    __syncthreads();
    for (uint32_t f = t; f < F; f += kOutThreads)
        if (p.ftot[f] > s_fstart[f + 1] - s_fstart[f]) s_bad = 1;
    __syncthreads();
    const bool bad = s_bad != 0;
    if (bad && blockIdx.x == 0 && t == 0) set_status(p.hdr, MMBEV_DEV_BOUNDS);
    {
        constexpr int per = kMaxFrames / kOutThreads;
        uint32_t c[per], sum = 0;
#pragma unroll
        for (int k = 0; k < per; ++k) {
            const uint32_t f = per * (uint32_t)t + k;
            const uint32_t u = f < F && !bad ? p.ftot[f] : 0u;
            c[k] = u <= maxv ? (u + kChunkRows - 1) / kChunkRows : 0u;
            sum += c[k];
            if (blockIdx.x == 0 && f < F) p.out_nvox[f] = (int32_t)min(u, maxv);
        }
        uint32_t tot = 0;
        uint32_t run = block_exclusive_scan(sum, s_warp, &tot);
#pragma unroll
        for (int k = 0; k < per; ++k) {
            const uint32_t f = per * (uint32_t)t + k;
            if (f < F) s_cpre[f] = run;
            run += c[k];
        }
        if (t == 0) s_cpre[F] = tot;
        __syncthreads();
    }
    const uint32_t C = s_cpre[F];
    for (uint32_t f = blockIdx.x; f < F && !bad; f += gridDim.x)   // block-uniform
        if (p.ftot[f] > maxv) capped_frame<B>(p, f, s_fstart[f], s_fstart[f + 1], s_hist, s_warp);
    for (uint32_t c = blockIdx.x; c < C; c += gridDim.x) {
        uint32_t lo = 0, hi = F;   // s_cpre[lo] <= c < s_cpre[hi]
        while (hi - lo > 1) {
            const uint32_t mid = (lo + hi) >> 1;
            if (s_cpre[mid] <= c) lo = mid; else hi = mid;
        }
        const uint32_t f = lo;
        const uint32_t row = (c - s_cpre[f]) * kChunkRows + (uint32_t)t;
        if (row < p.ftot[f]) emit_voxel<B>(p, f, row, s_fstart[f] + row, s_fstart[f], s_fstart[f + 1]);
    }
}

}  // namespace

cudaError_t launch_compact(const Params& p, int num_sms, bool pdl, cudaStream_t st) {
    (void)num_sms;   // a block per classify block
    static std::atomic<int> configured[64];
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    if (dev < 0 || dev >= 64 || !configured[dev].load(std::memory_order_acquire)) {
        e = cudaFuncSetAttribute(k_compact, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kCSmem);
        if (e != cudaSuccess) return e;
        if (dev >= 0 && dev < 64) configured[dev].store(1, std::memory_order_release);
    }
    return launch_k(k_compact, dim3(p.cls_grid > 0 ? p.cls_grid : 1u), dim3(kCT), kCSmem, st, pdl, p);
}

cudaError_t launch_sort(const Params& p, int num_sms, bool pdl, cudaStream_t st) {
    const uint32_t cap = (uint32_t)num_sms * 2u;
    const uint32_t g = p.sort_tiles_cap < cap ? p.sort_tiles_cap : cap;
    for (int pass = 0; pass < p.sort_passes; ++pass) {
        const bool to_b = (pass & 1) == 0;   // A -> B, B -> A, ...
        const cudaError_t e = launch_k(
            k_sort_pass, dim3(g > 0 ? g : 1u), dim3(kST), 0, st, pdl || pass > 0, p, pass,
            to_b ? p.key_a : p.key_b, to_b ? p.val_a : p.val_b, to_b ? p.key_b : p.key_a,
            to_b ? p.val_b : p.val_a);
        if (e != cudaSuccess) return e;
    }
    return cudaSuccess;
}

cudaError_t launch_runs(const Params& p, int num_sms, bool pdl, cudaStream_t st) {
    const uint32_t cap = (uint32_t)num_sms * 8u;
    const uint32_t g = p.run_tiles_cap < cap ? p.run_tiles_cap : cap;
    return launch_k(k_runs, dim3(g > 0 ? g : 1u), dim3(kRT), 0, st, pdl, p);
}

cudaError_t launch_emit(const Params& p, int num_sms, bool pdl, cudaStream_t st) {
    const dim3 grid(num_sms * (p.K <= 12 ? 6 : 2)), block(kOutThreads);
    if (p.K <= 4) return launch_k(k_emit<4>, grid, block, 0, st, pdl, p);
    if (p.K <= 12) return launch_k(k_emit<12>, grid, block, 0, st, pdl, p);
    if (p.K <= 32) return launch_k(k_emit<32>, grid, block, 0, st, pdl, p);
    return launch_k(k_emit<kMaxK>, grid, block, 0, st, pdl, p);
}

}  // namespace mmbev
