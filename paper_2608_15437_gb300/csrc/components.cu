// Voxel-grid connected components (the proposer of the paper's robot
// deployment, Sec. VI-F): occupied voxels of each frame joined under
// 26-connectivity.
//
// Union-find over each frame's kept rows. Rows ascend by linear index within
// a frame, so a voxel's neighbours with smaller rows are the 13 with a
// smaller index (the whole z-1 plane, then (y-1, x-1..x+1) and (y, x-1) of
// its own plane); each pair is joined once, from its larger row, by hooking
// the larger root under the smaller with a compare-and-swap (retried when
// another join moved a root meanwhile). Roots only ever hook under smaller
// rows, so every component ends rooted at its smallest row. Joins run as a
// warp-converged state machine (one parent-array step per lane per
// iteration), so the lanes' memory latencies overlap; walks split the path.
//
// Cluster path (per-frame caps up to 8 x 32,768 rows): one thread-block
// cluster per frame, the frame's rows split evenly over its CTAs, each CTA
// holding its rows' parents in its own shared memory. Neighbours are found
// by the row order itself: each CTA stages the linear indices of the rows
// its rows can reach (from one plane and line before its first row) in
// shared memory and binary-searches them. One launch runs the phases:
// parents; joins within the CTA, on its own shared memory; every row to its
// root within the CTA; the pairs reaching an earlier CTA (rows within one
// plane and line of the CTA's start), as pairs of those roots gathered in a
// set, one join per distinct pair through distributed shared memory;
// flatten (finds that only read, so a stale path-splitting store cannot
// overwrite a root already stored); labels, component sizes and boxes
// (pooled across the lanes of a warp that share a root).
//
// Multi-launch path (larger caps): five launches over a frame grid, the
// parent array being out_labels itself and neighbours found through a hash
// of (lin + 1) -> (row + 1) in the frame's own region of the caller's
// all-zero table: 16-byte buckets of two slots, the slots in use sized from
// the frame's kept voxels (4x, a power of two). Each inserting row records
// its slot in a scratch array past the slot regions; after every lookup of
// the frame has finished those slots and the scratch are zeroed, so the
// table is all-zero again.
#include <cooperative_groups.h>

#include <algorithm>
#include <atomic>
#include <climits>
#include <cstdint>

#include "mmbev_internal.cuh"

namespace cg = cooperative_groups;

namespace mmbev {
namespace {

constexpr int kCcThreads = 256;           // multi-launch path
constexpr int kClThreads = 1024;          // cluster path
constexpr int kClRowsMax = 32768;         // parents per CTA (128 KB)
constexpr int kClLinMax = 16384;          // linear indices of a CTA's window of rows (64 KB)
constexpr int kClSet = 2048;              // distinct pairs of roots across CTAs (16 KB)
constexpr int kClMaxCluster = 8;          // portable cluster size
constexpr uint32_t kUnionLimit = 1u << 20;
constexpr int32_t kMaxCcVoxels = 1 << 28; // keeps slot indices within 32 bits

struct CcArgs {
    const int32_t* coords;
    const int32_t* nvox;
    int32_t F, maxv, nx, ny, nz;
    uint2* slots;           // [F][hmax] {lin + 1, frame row + 1}; {0, 0}: empty
    uint32_t hmax;          // slots per frame region, a power of two >= 4 max_voxels
    uint32_t* slot_of;      // [F*max_voxels] slot + 1 the row inserted (0: none)
    int32_t* labels;        // out_labels
    int32_t* comp;          // [F*max_voxels][7] or null
    int32_t* ncomp;
    uint32_t* status;       // or null
};

__device__ __forceinline__ void cc_flag(const CcArgs& a, uint32_t bits) {
    if (a.status) atomicOr(a.status, bits);
}
__device__ __forceinline__ int cc_nv(const CcArgs& a, int f) {
    return min(max(__ldg(a.nvox + f), 0), a.maxv);
}
// Row g's coordinates, and whether they lie in the grid.
__device__ __forceinline__ bool cc_coords(const CcArgs& a, size_t g, int& z, int& y, int& x) {
    z = __ldg(a.coords + 3 * g);
    y = __ldg(a.coords + 3 * g + 1);
    x = __ldg(a.coords + 3 * g + 2);
    return z >= 0 && z < a.nz && y >= 0 && y < a.ny && x >= 0 && x < a.nx;
}
// Hash key of an in-grid cell: its linear index + 1 (never 0).
__device__ __forceinline__ uint32_t cc_key(const CcArgs& a, int z, int y, int x) {
    return ((uint32_t)z * (uint32_t)a.ny + (uint32_t)y) * (uint32_t)a.nx + (uint32_t)x + 1u;
}
__device__ __forceinline__ uint32_t cc_home(uint32_t mask, uint32_t key) {
    return slot_home(mask, (unsigned long long)key);
}
// Buckets in use in a frame's region, minus one: slots a power of two >= 4
// nv (at least 64), two slots a bucket.
__device__ __forceinline__ uint32_t cc_bmask(const CcArgs& a, int nv) {
    uint32_t h = 64;
    while (h < 4u * (uint32_t)nv && h < a.hmax) h <<= 1;
    return (h >> 1) - 1u;
}

// Insert (key -> v + 1) into the frame's buckets (the first free slot from
// the home bucket on); record the slot for the clear.
__device__ __forceinline__ void cc_insert(const CcArgs& a, uint2* reg, uint32_t bmask,
                                          uint32_t key, size_t g, int v) {
    uint32_t b = cc_home(bmask, key);
    for (uint32_t probe = 0; probe <= bmask; ++probe) {
        for (uint32_t s = 0; s < 2; ++s) {
            const uint32_t h = 2u * b + s;
            const uint32_t old = atomicCAS(&reg[h].x, 0u, key);
            if (old == 0u) {
                __stcg(&reg[h].y, (uint32_t)v + 1u);   // L2 only: no stale L1 line
                a.slot_of[g] = h + 1u;
                return;
            }
            if (old == key) return;   // a duplicate coordinate: the first row wins
        }
        b = (b + 1u) & bmask;
    }
    cc_flag(a, MMBEV_DEV_TABLE_FULL);
}

// Frame row stored under key, or -1, probing from bucket b on. Slots are
// only ever filled while keys go in, so a bucket with a free slot ends the
// search. Loads go through L1: lookups only run once every key is in (and
// no load of the table precedes them in the launch), and neighbouring
// voxels probe the same buckets.
__device__ __forceinline__ int32_t cc_lookup(const uint2* reg, uint32_t bmask, uint32_t key,
                                             uint32_t b) {
    for (uint32_t probe = 0; probe <= bmask; ++probe) {
        const uint4 q = __ldca(reinterpret_cast<const uint4*>(reg) + b);
        if (q.x == key) return (int32_t)q.y - 1;
        if (q.z == key) return (int32_t)q.w - 1;
        if (q.x == 0u || q.z == 0u) return -1;
        b = (b + 1u) & bmask;
    }
    return -1;
}

// Neighbour q (0..12) of (z, y, x) with a smaller linear index: the z-1
// plane (q < 9), then (y-1, x-1..x+1) and (y, x-1) of the voxel's plane.
__device__ __forceinline__ void cc_nbr(int q, int z, int y, int x, int& zz, int& yy, int& xx) {
    zz = q < 9 ? z - 1 : z;
    yy = q < 9 ? y + q / 3 - 1 : (q < 12 ? y - 1 : y);
    xx = q < 9 ? x + q % 3 - 1 : (q < 12 ? x + q - 10 : x - 1);
}

// The frame's unused rows [nv, max_voxels): label -1.
__device__ __forceinline__ void cc_fill_unused(const CcArgs& a, size_t base, int nv, int t0,
                                               int ts) {
    int32_t* lab = a.labels + base;
    const int head = min(a.maxv, (nv + 3) & ~3);
    for (int v = nv + t0; v < head; v += ts) lab[v] = -1;
    if ((reinterpret_cast<uintptr_t>(lab) & 15u) == 0) {
        int4* p4 = reinterpret_cast<int4*>(lab);
        for (int i = (head >> 2) + t0; i < (a.maxv >> 2); i += ts) p4[i] = make_int4(-1, -1, -1, -1);
        for (int v = max(head, a.maxv & ~3) + t0; v < a.maxv; v += ts) lab[v] = -1;
    } else {
        for (int v = head + t0; v < a.maxv; v += ts) lab[v] = -1;
    }
}

// Shared-memory accesses by state space: this CTA's shared memory, and
// another CTA's of the cluster (mapa gives its address).
__device__ __forceinline__ uint32_t smem_addr(const void* p) {
    return (uint32_t)__cvta_generic_to_shared(p);
}
__device__ __forceinline__ int32_t lds(uint32_t a) {
    int32_t v;
    asm volatile("ld.volatile.shared.b32 %0, [%1];" : "=r"(v) : "r"(a) : "memory");
    return v;
}
__device__ __forceinline__ void sts(uint32_t a, int32_t v) {
    asm volatile("st.volatile.shared.b32 [%0], %1;" ::"r"(a), "r"(v) : "memory");
}
__device__ __forceinline__ int32_t cas_s(uint32_t a, int32_t c, int32_t v) {
    int32_t o;
    asm volatile("atom.shared.cas.b32 %0, [%1], %2, %3;" : "=r"(o) : "r"(a), "r"(c), "r"(v) : "memory");
    return o;
}
__device__ __forceinline__ uint32_t mapa_rank(uint32_t a, uint32_t rank) {
    uint32_t d;
    asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(d) : "r"(a), "r"(rank));
    return d;
}
__device__ __forceinline__ int32_t ldc(uint32_t a) {
    int32_t v;
    asm volatile("ld.relaxed.cluster.shared::cluster.b32 %0, [%1];" : "=r"(v) : "r"(a) : "memory");
    return v;
}
__device__ __forceinline__ void stc(uint32_t a, int32_t v) {
    asm volatile("st.relaxed.cluster.shared::cluster.b32 [%0], %1;" ::"r"(a), "r"(v) : "memory");
}
__device__ __forceinline__ int32_t cas_c(uint32_t a, int32_t c, int32_t v) {
    int32_t o;
    asm volatile("atom.relaxed.cluster.shared::cluster.cas.b32 %0, [%1], %2, %3;"
                 : "=r"(o) : "r"(a), "r"(c), "r"(v) : "memory");
    return o;
}

// Parent arrays, indexed by frame row: out_labels of the frame (multi-launch
// path); this CTA's rows [v0, v0 + R) in its shared memory; the whole frame
// across the cluster, R rows per CTA.
struct GlobalPar {
    int32_t* p;
    __device__ __forceinline__ int32_t ld(int32_t x) const { return __ldcg(p + x); }
    __device__ __forceinline__ void st(int32_t x, int32_t v) const { p[x] = v; }
    __device__ __forceinline__ int32_t cas(int32_t x, int32_t c, int32_t v) const {
        return atomicCAS(p + x, c, v);
    }
};
struct LocalPar {
    uint32_t s;   // shared address of row v0's parent
    int32_t v0;
    __device__ __forceinline__ uint32_t at(int32_t x) const { return s + 4u * (uint32_t)(x - v0); }
    __device__ __forceinline__ int32_t ld(int32_t x) const { return lds(at(x)); }
    __device__ __forceinline__ void st(int32_t x, int32_t v) const { sts(at(x), v); }
    __device__ __forceinline__ int32_t cas(int32_t x, int32_t c, int32_t v) const {
        return cas_s(at(x), c, v);
    }
};
struct ClusterPar {
    uint32_t s;   // shared address of this CTA's first parent
    int32_t R;    // rows per CTA
    __device__ __forceinline__ uint32_t at(int32_t x) const {
        const int32_t r = x / R;
        return mapa_rank(s + 4u * (uint32_t)(x - r * R), (uint32_t)r);
    }
    __device__ __forceinline__ int32_t ld(int32_t x) const { return ldc(at(x)); }
    __device__ __forceinline__ void st(int32_t x, int32_t v) const { stc(at(x), v); }
    __device__ __forceinline__ int32_t cas(int32_t x, int32_t c, int32_t v) const {
        return cas_c(at(x), c, v);
    }
};

// Root of x, by reads only (the flatten pass: a stale path-splitting store
// could otherwise land after another thread stored a row's root).
template <class Par>
__device__ __forceinline__ int32_t uf_root(const CcArgs& a, const Par& P, int32_t x) {
    for (uint32_t i = 0; i < kUnionLimit; ++i) {
        const int32_t p = P.ld(x);
        if (p == x) return x;
        if (p < 0) {   // not a kept row: a table that was not clean
            cc_flag(a, MMBEV_DEV_BOUNDS);
            return x;
        }
        x = p;
    }
    cc_flag(a, MMBEV_DEV_WAIT_TIMEOUT);
    return x;
}

// The 13 neighbours of frame row v with a smaller index: nb[q] their rows,
// bit q of the result set for each one present (active: this lane holds an
// in-grid row at z, y, x). The home buckets are loaded together, through L1
// (see cc_lookup); the rare continuations (a home bucket full of other
// keys) follow.
__device__ __forceinline__ uint32_t cc_probe_row(const CcArgs& a, const uint2* reg,
                                                 uint32_t bmask, bool active, int v, int z,
                                                 int y, int x, int32_t nb[13],
                                                 uint32_t want = 0x1FFFu) {
    const uint4* bk = reinterpret_cast<const uint4*>(reg);
    uint32_t pend = 0;
    uint32_t cont = 0;   // bit q: its home bucket held two other keys
#pragma unroll
    for (int q = 0; q < 13; ++q) {
        int zz, yy, xx;
        cc_nbr(q, z, y, x, zz, yy, xx);
        const bool in = active && (want >> q & 1u) && zz >= 0 && zz < a.nz && yy >= 0 &&
                        yy < a.ny && xx >= 0 && xx < a.nx;
        const uint32_t k = cc_key(a, zz, yy, xx);
        const uint4 b = in ? __ldca(bk + cc_home(bmask, k)) : make_uint4(0u, 0u, 0u, 0u);
        const int32_t u = b.x == k ? (int32_t)b.y - 1 : (b.z == k ? (int32_t)b.w - 1 : -1);
        nb[q] = u;
        if (u >= 0 && u < v) pend |= 1u << q;   // u >= v: never for a clean table
        else if (in && u < 0 && b.x != 0u && b.z != 0u) cont |= 1u << q;
    }
    while (cont) {
        const int q = __ffs(cont) - 1;
        cont &= cont - 1u;
        int zz, yy, xx;
        cc_nbr(q, z, y, x, zz, yy, xx);
        const uint32_t k = cc_key(a, zz, yy, xx);
        const int32_t u = cc_lookup(reg, bmask, k, (cc_home(bmask, k) + 1u) & bmask);
        if (u >= 0 && u < v) {
            nb[q] = u;
            pend |= 1u << q;
        }
    }
    return pend;
}

// Join row me's set with the rows nb[q], q the set bits of pend. Whole
// warps call together. A state machine in which every lane takes exactly
// one step on the parent array per iteration (a read, or the hooking
// compare-and-swap), so the lanes' memory latencies overlap rather than add
// up; reads are plain loads, as many lanes read the same root word and
// atomics on one word serialize. Walks split the path: each node passed
// gets its grandparent, an ancestor, so concurrent walks and hooks stay
// valid.
template <class Par>
__device__ __forceinline__ void uf_join_all(const CcArgs& a, const Par& P, int32_t me,
                                            const int32_t* nb, uint32_t pend) {
    // stage 0: walk from me's set to its root ra; 1: walk from the neighbour
    // u to its root rb; 2: hook the larger root under the smaller; 3: done
    int32_t u = -1, cur = -1, prev = -1, ra = -1, rb = -1;
    int stage = 3;
    if (pend) {
        const int q = __ffs(pend) - 1;
        pend &= pend - 1u;
        u = nb[q];
        stage = 0;
        cur = me;
    }
    uint32_t steps = 0;
    while (__any_sync(0xFFFFFFFFu, stage != 3)) {
        if (++steps > kUnionLimit) {
            if (stage != 3) cc_flag(a, MMBEV_DEV_WAIT_TIMEOUT);
            break;
        }
        // this lane's one step: a read of cur's parent, or the hook
        const bool hook = stage == 2;
        const int32_t hi = ra > rb ? ra : rb, lo = ra > rb ? rb : ra;
        int32_t got = 0;
        if (hook) got = P.cas(hi, hi, lo);
        else if (stage != 3) got = P.ld(cur);
        bool edge_done = false;
        if (hook) {
            if (got == hi) {
                me = lo;
                edge_done = true;
            } else {   // another join moved a root: walk again from both roots
                stage = 0;
                cur = ra;
                prev = -1;
            }
        } else if (stage != 3) {
            if (got == cur || got < 0) {   // cur is a root (got < 0: a table that was not clean)
                if (got < 0) cc_flag(a, MMBEV_DEV_BOUNDS);
                if (stage == 0) {
                    ra = cur;
                    stage = 1;
                    cur = u;
                    prev = -1;
                } else {
                    rb = cur;
                    if (ra == rb) {
                        me = ra;
                        edge_done = true;
                    } else {
                        stage = 2;
                    }
                }
            } else {
                if (prev >= 0) P.st(prev, got);   // prev's grandparent
                prev = cur;
                cur = got;
            }
        }
        if (edge_done) {
            if (pend) {
                const int q = __ffs(pend) - 1;
                pend &= pend - 1u;
                u = nb[q];
                stage = 0;
                cur = me;
                prev = -1;
            } else {
                stage = 3;
            }
        }
    }
}

// Labels, component counts and boxes for one warp's rows (whole warps call
// together). root: the row's root, or -1.
__device__ __forceinline__ void cc_final_rows(const CcArgs& a, int f, size_t base, int v,
                                              bool valid, int32_t root, int z, int y, int x) {
    const int lane = threadIdx.x & 31;
    const unsigned roots = __ballot_sync(0xFFFFFFFFu, valid && root == v);
    if (lane == 0 && roots) atomicAdd(a.ncomp + f, __popc(roots));
    if (!a.comp) return;
    const int32_t key = valid ? root : -1 - lane;   // unique per idle lane: never pooled
    const unsigned peers = __match_any_sync(0xFFFFFFFFu, key);
    const int zmin = __reduce_min_sync(peers, z), zmax = __reduce_max_sync(peers, z);
    const int ymin = __reduce_min_sync(peers, y), ymax = __reduce_max_sync(peers, y);
    const int xmin = __reduce_min_sync(peers, x), xmax = __reduce_max_sync(peers, x);
    if (valid && lane == __ffs(peers) - 1) {
        int32_t* c = a.comp + 7 * (base + (size_t)root);
        atomicAdd(c, __popc(peers));
        atomicMin(c + 1, zmin); atomicMin(c + 2, ymin); atomicMin(c + 3, xmin);
        atomicMax(c + 4, zmax); atomicMax(c + 5, ymax); atomicMax(c + 6, xmax);
    }
}

__device__ __forceinline__ void cc_comp_init(const CcArgs& a, size_t g) {
    if (!a.comp) return;
    int32_t* c = a.comp + 7 * g;
    c[0] = 0;
    c[1] = c[2] = c[3] = INT_MAX;
    c[4] = c[5] = c[6] = INT_MIN;
}

// The slot row g inserted back to zero, and its scratch.
__device__ __forceinline__ void cc_clear_row(const CcArgs& a, uint2* reg, uint32_t bmask, size_t g) {
    const uint32_t h1 = a.slot_of[g];
    if (h1 == 0u) return;
    if (h1 - 1u <= 2u * bmask + 1u) reg[h1 - 1u] = make_uint2(0u, 0u);
    else cc_flag(a, MMBEV_DEV_BOUNDS);   // scratch that was not clean
    a.slot_of[g] = 0u;
}

// Join (ra, rb) one lane at a time (rare: a full set of root pairs).
__device__ __noinline__ void uf_join_lane(const CcArgs& a, const ClusterPar& G, int32_t ra,
                                          int32_t rb) {
    for (uint32_t i = 0; i < kUnionLimit; ++i) {
        ra = uf_root(a, G, ra);
        rb = uf_root(a, G, rb);
        if (ra == rb) return;
        const int32_t hi = ra > rb ? ra : rb, lo = ra > rb ? rb : ra;
        if (G.cas(hi, hi, lo) == hi) return;
    }
    cc_flag(a, MMBEV_DEV_WAIT_TIMEOUT);
}

// Linear index of an in-grid cell.
__device__ __forceinline__ uint32_t cc_lin(const CcArgs& a, int z, int y, int x) {
    return ((uint32_t)z * (uint32_t)a.ny + (uint32_t)y) * (uint32_t)a.nx + (uint32_t)x;
}
// Linear index of frame row i: from a window of rows [lo, ...) held in
// shared memory, or from the coordinates in global memory.
struct SmemLins {
    const uint32_t* s;
    int lo;
    __device__ __forceinline__ uint32_t operator()(int i) const { return s[i - lo]; }
};
struct GlobalLins {
    const CcArgs* a;
    size_t base;
    __device__ __forceinline__ uint32_t operator()(int i) const {
        const size_t g = base + (size_t)i;
        return cc_lin(*a, __ldg(a->coords + 3 * g), __ldg(a->coords + 3 * g + 1),
                      __ldg(a->coords + 3 * g + 2));
    }
};

// First row of [lo, hi) whose linear index is >= t (rows ascend).
template <class Lins>
__device__ __forceinline__ int cc_lower_bound(const Lins& S, int lo, int hi, long long t) {
    while (lo < hi) {
        const int mid = (lo + hi) >> 1;
        if ((long long)S(mid) < t) lo = mid + 1;
        else hi = mid;
    }
    return lo;
}

// The 13 neighbours of frame row v (in-grid at z, y, x, linear index lv)
// with a smaller linear index, found among rows [lo, v) by their order:
// in each of the lines (z-1, y-1), (z-1, y), (z-1, y+1) and (z, y-1) a
// binary search for the cell at x-1, then at most three rows in turn; the
// cell (z, y, x-1) is row v-1 when present. nb[q] their rows (q numbered as
// in cc_nbr), bit q of the result set for each one present.
template <class Lins>
__device__ __forceinline__ uint32_t cc_search_row(const CcArgs& a, const Lins& S, int lo, int v,
                                                  int z, int y, int x, uint32_t lv,
                                                  int32_t nb[13]) {
    uint32_t pend = 0;
    int from = lo;
#pragma unroll
    for (int g = 0; g < 4; ++g) {
        const int dz = g < 3 ? -1 : 0, dy = g < 3 ? g - 1 : -1;
        if (z + dz < 0 || y + dy < 0 || y + dy >= a.ny) continue;
        const long long c = (long long)lv + ((long long)dz * a.ny + dy) * (long long)a.nx;
        int j = cc_lower_bound(S, from, v, c - 1);
        from = j;
#pragma unroll
        for (int dx = -1; dx <= 1; ++dx) {
            const long long t = c + dx;
            while (j < v && (long long)S(j) < t) ++j;
            if (x + dx >= 0 && x + dx < a.nx && j < v && (long long)S(j) == t) {
                nb[3 * g + dx + 1] = j;
                pend |= 1u << (3 * g + dx + 1);
            }
        }
    }
    if (x > 0 && v - 1 >= lo && S(v - 1) == lv - 1u) {
        nb[12] = v - 1;
        pend |= 1u << 12;
    }
    return pend;
}

// Row v of this CTA (in-grid at z, y, x, linear index lv), once every row
// points at its root within its CTA: its pairs reaching an earlier CTA as
// pairs of those roots, into the set of distinct pairs. Loads are
// independent across positions, so they overlap.
template <class Lins>
__device__ __forceinline__ void cc_far_row(const CcArgs& a, const LocalPar& L,
                                           const ClusterPar& G, const Lins& S, int lo, int v,
                                           int z, int y, int x, uint32_t lv,
                                           unsigned long long* set) {
    int32_t nb[13];
    const uint32_t pend = cc_search_row(a, S, lo, v, z, y, x, lv, nb);
    const int32_t ra = L.ld(v);
    int32_t rb[13];
#pragma unroll
    for (int q = 0; q < 13; ++q) rb[q] = (pend >> q & 1u) && nb[q] < L.v0 ? G.ld(nb[q]) : -1;
#pragma unroll 1
    for (int q = 0; q < 13; ++q) {
        if (rb[q] < 0 || ra < 0 || rb[q] == ra) continue;
        const int32_t hi = ra > rb[q] ? ra : rb[q], lo2 = ra > rb[q] ? rb[q] : ra;
        const unsigned long long key = ((unsigned long long)(uint32_t)hi << 32) | (uint32_t)lo2;
        uint32_t h = (uint32_t)mix64(key) & (kClSet - 1);
        bool placed = false;
        for (int probe = 0; probe < kClSet; ++probe) {
            const unsigned long long old = atomicCAS(set + h, 0ull, key);
            if (old == 0ull || old == key) {
                placed = true;
                break;
            }
            h = (h + 1u) & (kClSet - 1);
        }
        if (!placed) uf_join_lane(a, G, hi, lo2);
    }
}

// First row of [0, n) whose linear index is >= T, for a frame whose rows
// ascend: two rounds of loads spread over the CTA's threads (samples every
// ceil(n / threads) rows, then the rows between two samples). All threads
// of the CTA call together.
__device__ __forceinline__ int cc_window_lo(const CcArgs& a, size_t base, int n, long long T) {
    if (n == 0 || T <= 0) return 0;
    const GlobalLins S{&a, base};
    const int step = (n + kClThreads - 1) / kClThreads;
    const int r = (int)threadIdx.x * step;
    const int c1 = __syncthreads_count(r < n && (long long)S(r) < T);
    if (c1 == 0) return 0;
    const int b2 = (c1 - 1) * step + 1;
    const int e2 = min(c1 * step, n);
    const int r2 = b2 + (int)threadIdx.x;
    const int c2 = __syncthreads_count(r2 < e2 && (long long)S(r2) < T);
    return b2 + c2;
}

// ---------------------------------------------------------------- cluster path

template <class Lins>
__device__ __forceinline__ void cc_cluster_joins(const CcArgs& a, const Lins& S, int lo, int f,
                                                 int nv, int v0, int v1, int R, int32_t* s_par,
                                                 unsigned long long* s_set, int* s_next) {
    cg::cluster_group cl = cg::this_cluster();
    const size_t base = (size_t)f * (size_t)a.maxv;
    const int t = threadIdx.x, lane = t & 31;
    const LocalPar L{smem_addr(s_par), v0};

    // 2. joins within this CTA's rows, on its own shared memory; each warp
    // takes the next 32 rows from a shared counter (join chains vary in
    // length), and pairs reaching an earlier CTA wait
    for (;;) {
        int w0 = 0;
        if (lane == 0) w0 = atomicAdd(s_next, 32);
        w0 = __shfl_sync(0xFFFFFFFFu, w0, 0);
        if (w0 >= v1) break;
        const int v = w0 + lane;
        int z = 0, y = 0, x = 0;
        const bool active = v < v1 && cc_coords(a, base + (size_t)v, z, y, x);
        int32_t nb[13];
        uint32_t pend = 0;
        if (active) pend = cc_search_row(a, S, lo, v, z, y, x, cc_lin(a, z, y, x), nb);
        uint32_t far = 0;
#pragma unroll
        for (int q = 0; q < 13; ++q)
            if ((pend >> q & 1u) && nb[q] < v0) far |= 1u << q;
        uf_join_all(a, L, v, nb, pend & ~far);
    }
    __syncthreads();

    // 3. every row to its root within this CTA (joins so far stay within a
    // CTA, so these roots are final until the pairs below)
    for (int v = v0 + t; v < v1; v += kClThreads) {
        const int32_t p = s_par[v - v0];
        if (p < 0 || p == v) continue;
        int32_t r = p;
        for (uint32_t i = 0; i < kUnionLimit; ++i) {
            const int32_t q = L.ld(r);
            if (q == r || q < 0) break;
            r = q;
        }
        L.st(v, r);
    }
    cl.sync();

    // 4. the pairs reaching an earlier CTA (only rows within one plane and
    // line of the CTA's first row have any), as pairs of roots (v's in this
    // CTA, u's in its own) gathered in a set; then one join per distinct
    // pair, through the cluster
    const ClusterPar G{smem_addr(s_par), R};
    if (lo < v0 && v0 < v1) {   // rows [lo, v0) exist: row v0 - 1 is in the window
        const long long reach = (long long)S(v0 - 1) + (long long)a.ny * a.nx + a.nx + 1;
        for (int v = v0 + t; v < v1; v += kClThreads) {
            int z, y, x;
            if (!cc_coords(a, base + (size_t)v, z, y, x)) continue;
            const uint32_t lv = cc_lin(a, z, y, x);
            if ((long long)lv > reach) break;   // rows ascend: none further on either
            cc_far_row(a, L, G, S, lo, v, z, y, x, lv, s_set);
        }
    }
    __syncthreads();
    for (int e0 = t & ~31; e0 < kClSet; e0 += kClThreads) {
        const unsigned long long key = s_set[e0 + lane];
        const int32_t hi = (int32_t)(key >> 32), lo2 = (int32_t)(uint32_t)key;
        uf_join_all(a, G, hi, &lo2, key ? 1u : 0u);
    }
    cl.sync();

    // 5. every row to its root (finds that only read)
    for (int v = v0 + t; v < v1; v += kClThreads) {
        const int32_t p = s_par[v - v0];
        if (p >= 0 && p != v) s_par[v - v0] = uf_root(a, G, p);
    }
    cl.sync();
}

__global__ void __launch_bounds__(kClThreads, 1) k_cc_cluster(CcArgs a, int C, int rcap) {
    // [kClSet] distinct pairs of roots, [rcap] parents, [kClLinMax] linear
    // indices of the rows [lo, v1)
    extern __shared__ unsigned long long s_dyn[];
    __shared__ int s_next;   // the next row of the join phase
    unsigned long long* s_set = s_dyn;
    int32_t* s_par = reinterpret_cast<int32_t*>(s_dyn + kClSet);
    uint32_t* s_lin = reinterpret_cast<uint32_t*>(s_par + rcap);
    cg::cluster_group cl = cg::this_cluster();
    const int rank = (int)cl.block_rank();
    const int f = blockIdx.x / C;
    const int nv = cc_nv(a, f);
    const int R = max(1, (nv + C - 1) / C);   // <= rcap, as nv <= max_voxels
    const int v0 = min(nv, rank * R), v1 = min(nv, v0 + R);
    const size_t base = (size_t)f * (size_t)a.maxv;
    const int t = threadIdx.x, lane = t & 31;
    if (rank == 0 && t == 0) a.ncomp[f] = 0;
    if (t == 0) s_next = v0;
    for (int i = t; i < kClSet; i += kClThreads) s_set[i] = 0ull;

    // the window of rows any of this CTA's rows may neighbour: from the
    // first row at or past (linear index of v0) - (nx ny + nx + 1)
    const GlobalLins GL{&a, base};
    long long T = 0;
    if (v0 < v1) T = (long long)GL(v0) - ((long long)a.ny * a.nx + a.nx + 1);
    const int lo = v0 < v1 ? cc_window_lo(a, base, v0, T) : v0;
    const bool in_smem = v1 - lo <= kClLinMax;
    if (in_smem)
        for (int i = lo + t; i < v1; i += kClThreads) s_lin[i - lo] = GL(i);

    // 1. every kept row its own root; rows must ascend by linear index
    for (int v = v0 + t; v < v1; v += kClThreads) {
        const size_t g = base + (size_t)v;
        int z, y, x;
        if (!cc_coords(a, g, z, y, x)) {
            s_par[v - v0] = -1;
            continue;
        }
        s_par[v - v0] = v;
        cc_comp_init(a, g);
        if (v > 0 && GL(v - 1) >= cc_lin(a, z, y, x)) cc_flag(a, MMBEV_DEV_UNSORTED);
    }
    cc_fill_unused(a, base, nv, rank * kClThreads + t, C * kClThreads);
    __syncthreads();

    if (in_smem) cc_cluster_joins(a, SmemLins{s_lin, lo}, lo, f, nv, v0, v1, R, s_par, s_set, &s_next);
    else cc_cluster_joins(a, GL, lo, f, nv, v0, v1, R, s_par, s_set, &s_next);

    // 6. labels, components (this CTA's rows only: no other CTA's memory is
    // touched past the last barrier)
    for (int w0 = v0 + (t & ~31); w0 < v1; w0 += kClThreads) {
        const int v = w0 + lane;
        int z = 0, y = 0, x = 0;
        bool valid = false;
        int32_t root = -1;
        if (v < v1) {
            const size_t g = base + (size_t)v;
            root = s_par[v - v0];
            valid = root >= 0 && cc_coords(a, g, z, y, x);
            a.labels[g] = valid ? root : -1;
        }
        cc_final_rows(a, f, base, v, valid, root, z, y, x);
    }
}

// ---------------------------------------------------------------- multi-launch path

__global__ void __launch_bounds__(kCcThreads) k_cc_insert(CcArgs a) {
    const int f = blockIdx.y;
    const int nv = cc_nv(a, f);
    const size_t base = (size_t)f * (size_t)a.maxv;
    uint2* reg = a.slots + (size_t)f * a.hmax;
    const uint32_t bmask = cc_bmask(a, nv);
    const int t0 = blockIdx.x * blockDim.x + threadIdx.x, ts = gridDim.x * blockDim.x;
    if (t0 == 0) a.ncomp[f] = 0;
    for (int v = t0; v < nv; v += ts) {
        const size_t g = base + (size_t)v;
        int z, y, x;
        if (!cc_coords(a, g, z, y, x)) {
            a.labels[g] = -1;
            continue;
        }
        a.labels[g] = v;
        cc_comp_init(a, g);
        cc_insert(a, reg, bmask, cc_key(a, z, y, x), g, v);
    }
    cc_fill_unused(a, base, nv, t0, ts);
}

__global__ void __launch_bounds__(kCcThreads, 4) k_cc_link(CcArgs a) {
    pdl_wait();
    const int f = blockIdx.y;
    const int nv = cc_nv(a, f);
    const size_t base = (size_t)f * (size_t)a.maxv;
    const GlobalPar P{a.labels + base};
    const uint2* reg = a.slots + (size_t)f * a.hmax;
    const uint32_t bmask = cc_bmask(a, nv);
    const int lane = threadIdx.x & 31;
    for (int w0 = blockIdx.x * blockDim.x + (threadIdx.x & ~31); w0 < nv;
         w0 += gridDim.x * blockDim.x) {   // whole warps iterate together
        const int v = w0 + lane;
        int z = 0, y = 0, x = 0;
        const bool active = v < nv && cc_coords(a, base + (size_t)v, z, y, x);
        int32_t nb[13];
        const uint32_t pend = cc_probe_row(a, reg, bmask, active, v, z, y, x, nb);
        uf_join_all(a, P, v, nb, pend);
    }
}

__global__ void __launch_bounds__(kCcThreads) k_cc_flatten(CcArgs a) {
    pdl_wait();
    const int f = blockIdx.y;
    const int nv = cc_nv(a, f);
    const GlobalPar P{a.labels + (size_t)f * (size_t)a.maxv};
    for (int v = blockIdx.x * blockDim.x + threadIdx.x; v < nv; v += gridDim.x * blockDim.x) {
        const int32_t p = P.ld(v);
        if (p >= 0 && p != v) P.st(v, uf_root(a, P, p));
    }
}

__global__ void __launch_bounds__(kCcThreads) k_cc_final(CcArgs a) {
    pdl_wait();
    const int f = blockIdx.y;
    const int nv = cc_nv(a, f);
    const size_t base = (size_t)f * (size_t)a.maxv;
    const int lane = threadIdx.x & 31;
    // whole warps iterate together (the stride and each warp's start are
    // multiples of 32)
    for (int w0 = blockIdx.x * blockDim.x + (threadIdx.x & ~31); w0 < nv;
         w0 += gridDim.x * blockDim.x) {
        const int v = w0 + lane;
        int z = 0, y = 0, x = 0;
        bool valid = false;
        int32_t root = -1;
        if (v < nv) {
            root = a.labels[base + v];
            valid = root >= 0 && cc_coords(a, base + (size_t)v, z, y, x);
        }
        cc_final_rows(a, f, base, v, valid, root, z, y, x);
    }
}

// After every lookup: the slots the kept rows inserted, and the scratch,
// back to zero.
__global__ void __launch_bounds__(kCcThreads) k_cc_clear(CcArgs a) {
    pdl_wait();
    const int f = blockIdx.y;
    const int nv = cc_nv(a, f);
    const size_t base = (size_t)f * (size_t)a.maxv;
    uint2* reg = a.slots + (size_t)f * a.hmax;
    const uint32_t bmask = cc_bmask(a, nv);
    for (int v = blockIdx.x * blockDim.x + threadIdx.x; v < nv; v += gridDim.x * blockDim.x)
        cc_clear_row(a, reg, bmask, base + (size_t)v);
}

// Slots per frame region for a per-frame cap: a power of two >= 4 cap, >= 64.
unsigned long long cc_hmax(long long max_voxels) {
    unsigned long long h = 64;
    while (h < 4ull * (unsigned long long)max_voxels) h <<= 1;
    return h;
}

// Cluster size for this launch, or 0 for the multi-launch path; the rows of
// parents per CTA (even) in *rcap.
int cc_cluster_size(int num_frames, int max_voxels, int sms, int* rcap) {
    const int cmin = (int)(((long long)max_voxels + kClRowsMax - 1) / kClRowsMax);
    if (cmin > kClMaxCluster) return 0;
    const int cpar = std::max(1, std::min(kClMaxCluster, sms / std::max(1, num_frames)));
    const int C = std::max(std::max(cmin, 1), cpar);
    *rcap = (int)((((long long)max_voxels + C - 1) / C + 1) & ~1ll);
    return C;
}

}  // namespace
}  // namespace mmbev

using namespace mmbev;

extern "C" size_t mmbev_components_table_size(int32_t num_frames, int32_t max_voxels) {
    if (num_frames < 0 || num_frames > kMaxFrames || max_voxels < 0 || max_voxels > kMaxCcVoxels)
        return 0;
    if (max_voxels <= kClMaxCluster * kClRowsMax) return 0;   // the cluster path needs none
    const unsigned long long rows = (unsigned long long)num_frames * (unsigned long long)max_voxels;
    return (size_t)((unsigned long long)num_frames * cc_hmax(max_voxels) * sizeof(uint2) +
                     rows * sizeof(uint32_t));
}

extern "C" int mmbev_voxel_components(const int32_t* coords, const int32_t* nvox,
                                      int32_t num_frames, int32_t max_voxels,
                                      const int32_t dims[3], void* table, size_t table_bytes,
                                      int32_t* out_labels, int32_t* out_comp,
                                      int32_t* out_ncomp, uint32_t* out_status,
                                      cudaStream_t stream) {
    if (num_frames < 0 || num_frames > kMaxFrames || max_voxels < 0 || !dims) return MMBEV_EINVAL;
    if (max_voxels > kMaxCcVoxels) return MMBEV_EINVAL;
    if (dims[0] < 1 || dims[1] < 1 || dims[2] < 1) return MMBEV_EINVAL;
    if ((unsigned long long)dims[0] * dims[1] * dims[2] > 0xFFFFFFFFull) return MMBEV_EINVAL;
    const unsigned long long rows = (unsigned long long)num_frames * (unsigned long long)max_voxels;
    if (rows == 0) return MMBEV_OK;
    if (rows > 0x7FFFFFFFull) return MMBEV_EINVAL;
    if (!coords || !nvox || !out_labels || !out_ncomp) return MMBEV_EINVAL;
    const bool multi = max_voxels > kClMaxCluster * kClRowsMax;   // else no table is used
    if (multi) {
        if (!table || (reinterpret_cast<uintptr_t>(table) & 15u)) return MMBEV_EINVAL;
        if (mmbev_components_table_size(num_frames, max_voxels) > table_bytes)
            return MMBEV_EWORKSPACE;
    }
    int dev = 0, sms = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) return MMBEV_ECUDA;
    if (cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess)
        return MMBEV_ECUDA;
    CcArgs a;
    a.coords = coords;
    a.nvox = nvox;
    a.F = num_frames;
    a.maxv = max_voxels;
    a.nx = dims[0];
    a.ny = dims[1];
    a.nz = dims[2];
    a.hmax = (uint32_t)cc_hmax(max_voxels);
    a.slots = static_cast<uint2*>(table);
    a.slot_of = reinterpret_cast<uint32_t*>(a.slots + (size_t)num_frames * a.hmax);
    a.labels = out_labels;
    a.comp = out_comp;
    a.ncomp = out_ncomp;
    a.status = out_status;
    if (out_status && cudaMemsetAsync(out_status, 0, sizeof(uint32_t), stream) != cudaSuccess)
        return MMBEV_ECUDA;

    int rcap = 0;
    const int C = multi ? 0 : cc_cluster_size(num_frames, max_voxels, sms, &rcap);
    if (C > 0) {
        constexpr int kSmemMax = (int)(sizeof(unsigned long long) * kClSet +
                                       sizeof(int32_t) * kClRowsMax + sizeof(uint32_t) * kClLinMax);
        // raise the shared memory limit once per device (outside any capture)
        static std::atomic<int> configured[64];
        if (dev < 0 || dev >= 64 || !configured[dev].load(std::memory_order_acquire)) {
            if (cudaFuncSetAttribute(k_cc_cluster, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                     kSmemMax) != cudaSuccess)
                return MMBEV_ECUDA;
            if (dev >= 0 && dev < 64) configured[dev].store(1, std::memory_order_release);
        }
        cudaLaunchConfig_t cfg = {};
        cfg.gridDim = dim3((unsigned)(num_frames * C));
        cfg.blockDim = dim3(kClThreads);
        cfg.dynamicSmemBytes = sizeof(unsigned long long) * kClSet + sizeof(int32_t) * (size_t)rcap +
                               sizeof(uint32_t) * kClLinMax;
        cfg.stream = stream;
        cudaLaunchAttribute attr[1];
        attr[0].id = cudaLaunchAttributeClusterDimension;
        attr[0].val.clusterDim.x = (unsigned)C;
        attr[0].val.clusterDim.y = 1;
        attr[0].val.clusterDim.z = 1;
        cfg.attrs = attr;
        cfg.numAttrs = 1;
        return cudaLaunchKernelEx(&cfg, k_cc_cluster, a, C, rcap) == cudaSuccess ? MMBEV_OK
                                                                                 : MMBEV_ECUDA;
    }

    // a frame per grid row; together about 8 blocks per SM, each frame's
    // blocks striding over its kept rows
    const unsigned per_frame = (unsigned)std::max<long long>(
        1, std::min<long long>(((long long)max_voxels + kCcThreads - 1) / kCcThreads,
                               ((long long)sms * 8 + num_frames - 1) / num_frames));
    const dim3 grid(per_frame, (unsigned)num_frames), block(kCcThreads);
    cudaError_t e = launch_k(k_cc_insert, grid, block, 0, stream, false, a);
    if (e == cudaSuccess) e = launch_k(k_cc_link, grid, block, 0, stream, true, a);
    if (e == cudaSuccess) e = launch_k(k_cc_flatten, grid, block, 0, stream, true, a);
    if (e == cudaSuccess) e = launch_k(k_cc_final, grid, block, 0, stream, true, a);
    if (e == cudaSuccess) e = launch_k(k_cc_clear, grid, block, 0, stream, true, a);
    return e == cudaSuccess ? MMBEV_OK : MMBEV_ECUDA;
}
