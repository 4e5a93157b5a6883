// Host side of libmmbev: argument validation, workspace layout, and the
// fixed, stream-ordered launch sequence of the path. Nothing here allocates,
// synchronizes or keeps state across calls.
#include <cmath>
#include <cstring>
#include <atomic>

#include <vector>

#include "mmbev_internal.cuh"

namespace mmbev {
namespace {

constexpr size_t kAlign = 256;

size_t align_up(size_t x, size_t a) { return (x + a - 1) / a * a; }

struct Grid {
    uint32_t dims[3];
    uint64_t cells;
};

bool make_grid(const float* vs, const float* range, Grid* g) {
    if (!vs || !range) return false;
    uint64_t cells = 1;
    for (int a = 0; a < 3; ++a) {
        if (!std::isfinite(vs[a]) || !(vs[a] > 0.0f)) return false;
        if (!std::isfinite(range[a]) || !std::isfinite(range[a + 3])) return false;
        if (!(range[a + 3] > range[a])) return false;
        const double n = std::llround(((double)range[a + 3] - (double)range[a]) / (double)vs[a]);
        if (!(n >= 1.0) || n > 4294967295.0) return false;
        g->dims[a] = (uint32_t)n;
        cells *= (uint64_t)n;
        if (cells > 0xFFFFFFFFull) return false;
    }
    g->cells = cells;
    return true;
}

int mask_words_for(int32_t max_rois_frame) {
    const int w = (max_rois_frame + 31) / 32;
    return w < 1 ? 1 : w;
}

// Coarse candidate grid: G x G cells with G the largest even number (at most
// 64) whose mask of G^2 * mask_words words fits the classify kernel's
// shared-memory room per staged frame: 8,192 words (32 KB) up to 64 ROIs a
// frame, 4,096 words beyond, where the staged ROI tables grow. Even G keeps
// each frame's mask a whole number of 16-byte vectors.
int coarse_for(int mask_words) {
    const int w = mask_words < 1 ? 1 : mask_words;
    const int room = w <= 2 ? 8192 : 4096;
    int g = 64;
    while (g > 8 && g * g * w > room) g -= 2;
    return g;
}

// Byte offsets of every workspace array for one call shape.
struct Layout {
    size_t hdr, sweep_off, sweep_frame, fso, fro, roi_prep, masks;
    size_t records, ckey, key_a, val_a, rcnt, cls_cnt, cls_flo, fcnt, ftot, hist, sort_state,
        run_state, vdesc;
    size_t total;
    uint32_t num_tiles, sort_tiles_cap, run_tiles_cap;
    int mask_words, coarse;
};

Layout make_layout(int64_t max_points, int64_t rois_total, int32_t max_rois_frame,
                   int32_t max_voxels, int32_t num_frames, const Grid& g) {
    Layout L{};
    (void)g;
    L.mask_words = mask_words_for(max_rois_frame);
    L.coarse = coarse_for(L.mask_words);
    const size_t F = (size_t)num_frames, R = (size_t)(rois_total > 0 ? rois_total : 1);
    const size_t U = (size_t)(max_points > 0 ? max_points : 1);
    L.num_tiles = (uint32_t)((U + kTile - 1) / kTile);
    const size_t TS = (size_t)L.num_tiles * kTile;        // record slots, tile-aligned
    const size_t regions = TS / kRegion;
    // a frame's items are tiled from its own first item: at most one more
    // tile a frame than the call's items fill
    L.sort_tiles_cap = (uint32_t)((TS + kSortTile - 1) / kSortTile + F);
    L.run_tiles_cap = (uint32_t)((TS + kRunTile - 1) / kRunTile + F);
    size_t o = 0;
    auto take = [&](size_t bytes) { const size_t at = o; o = align_up(o + bytes, kAlign); return at; };
    L.hdr = take(sizeof(Header));
    L.sweep_off = take(sizeof(int64_t) * (kMaxSweeps + 1));
    L.sweep_frame = take(sizeof(int32_t) * kMaxSweeps);
    L.fso = take(sizeof(int32_t) * (F + 1));
    L.fro = take(sizeof(int32_t) * (F + 1));
    L.roi_prep = take(sizeof(RoiPrep) * R);
    // room for the largest mask any call with at most max_rois_frame ROIs per
    // frame selects (fewer ROIs can pick a finer grid), so the size is
    // monotone in max_rois_frame
    size_t mask_words_frame = 0;
    for (int w = 1; w <= L.mask_words; ++w) {
        const size_t c = (size_t)coarse_for(w);
        if (c * c * (size_t)w > mask_words_frame) mask_words_frame = c * c * (size_t)w;
    }
    L.masks = take(sizeof(uint32_t) * F * mask_words_frame);
    L.records = take(32 * TS);
    L.ckey = take(sizeof(unsigned long long) * TS);   // then sort buffer B: lins, positions
    L.key_a = take(sizeof(uint32_t) * TS);
    L.val_a = take(sizeof(uint32_t) * TS);
    L.rcnt = take(regions);
    L.cls_cnt = take(sizeof(uint32_t) * kMaxClsGrid);
    L.cls_flo = take(sizeof(uint32_t) * kMaxClsGrid);
    L.fcnt = take(sizeof(uint32_t) * F);
    L.ftot = take(sizeof(uint32_t) * F);
    L.hist = take(sizeof(uint32_t) * F * kMaxPasses * kDigits);
    L.sort_state = take(sizeof(unsigned long long) * 2 * (size_t)L.sort_tiles_cap * kDigits);
    L.run_state = take(sizeof(unsigned long long) * ((size_t)L.run_tiles_cap + 1));
    L.vdesc = take(sizeof(uint4) * TS);
    L.total = o;
    (void)max_voxels;
    return L;
}

// Validation shared by the full path and the classify-only path. Fills the
// call-shape fields of Params and the host descriptor.
int validate_common(const float* points, const int64_t* sweep_offsets, int32_t num_sweeps,
                    const float* sweep_tf, const mmbev_roi_t* rois, int32_t num_rois,
                    float roi_margin, const float* voxel_size, const float* range,
                    int32_t num_frames, const int32_t* fso, const int32_t* fro,
                    Params* p, HostDesc* d, Grid* g, int32_t* max_rois_frame) {
    if (num_sweeps < 0 || num_sweeps > kMaxSweeps) return MMBEV_EINVAL;
    if (num_frames < 1 || num_frames > kMaxFrames) return MMBEV_EINVAL;
    if (num_rois < 0) return MMBEV_EINVAL;
    if (!sweep_offsets || !fso || !fro) return MMBEV_EINVAL;
    if (!make_grid(voxel_size, range, g)) return MMBEV_EINVAL;
    if (!std::isfinite(roi_margin) || !(roi_margin >= 0.0f)) return MMBEV_EINVAL;
    if (sweep_offsets[0] != 0) return MMBEV_EINVAL;
    for (int s = 0; s < num_sweeps; ++s)
        if (sweep_offsets[s + 1] < sweep_offsets[s]) return MMBEV_EINVAL;
    const int64_t n = sweep_offsets[num_sweeps];
    if (n < 0 || n > kMaxPoints) return MMBEV_EINVAL;
    if (fso[0] != 0 || fso[num_frames] != num_sweeps) return MMBEV_EINVAL;
    if (fro[0] != 0 || fro[num_frames] != num_rois) return MMBEV_EINVAL;
    int32_t rmax = 0;
    for (int f = 0; f < num_frames; ++f) {
        if (fso[f + 1] < fso[f] || fro[f + 1] < fro[f]) return MMBEV_EINVAL;
        const int32_t rn = fro[f + 1] - fro[f];
        if (rn > kMaxRoisPerFrame) return MMBEV_EINVAL;
        if (rn > rmax) rmax = rn;
    }
    if (n > 0 && (!points || (reinterpret_cast<uintptr_t>(points) & 15u))) return MMBEV_EINVAL;
    if (num_sweeps > 0 && !sweep_tf) return MMBEV_EINVAL;
    if (num_rois > 0 && !rois) return MMBEV_EINVAL;

    std::memset(d, 0, sizeof(HostDesc));
    for (int s = 0; s <= num_sweeps; ++s) d->sweep_off[s] = sweep_offsets[s];
    for (int f = 0; f <= num_frames; ++f) {
        d->frame_sweep_off[f] = fso[f];
        d->frame_roi_off[f] = fro[f];
    }
    *p = Params{};
    p->points = points;
    p->sweep_tf = sweep_tf;
    p->rois = rois;
    p->num_points = n;
    p->num_sweeps = num_sweeps;
    p->num_frames = num_frames;
    p->num_rois = num_rois;
    p->margin = roi_margin;
    for (int a = 0; a < 3; ++a) {
        p->vs[a] = voxel_size[a];
        p->rmin[a] = range[a];
        p->rmax[a] = range[a + 3];
        p->dims[a] = g->dims[a];
    }
    p->cells = (uint32_t)g->cells;
    {
        // 9-bit digits of the largest lin
        const uint64_t maxlin = g->cells - 1ull;
        int bits = 0;
        while (bits < 64 && (maxlin >> bits) != 0ull) ++bits;
        p->sort_passes = (bits + kDigitBits - 1) / kDigitBits;
    }
    p->div_nx = udiv_make(g->dims[0]);
    p->div_ny = udiv_make(g->dims[1]);
    *max_rois_frame = rmax;
    return MMBEV_OK;
}

void bind_layout(Params* p, const Layout& L, uint8_t* ws) {
    p->hdr = reinterpret_cast<Header*>(ws + L.hdr);
    p->sweep_off = reinterpret_cast<int64_t*>(ws + L.sweep_off);
    p->sweep_frame = reinterpret_cast<int32_t*>(ws + L.sweep_frame);
    p->frame_sweep_off = reinterpret_cast<int32_t*>(ws + L.fso);
    p->frame_roi_off = reinterpret_cast<int32_t*>(ws + L.fro);
    p->roi_prep = reinterpret_cast<RoiPrep*>(ws + L.roi_prep);
    p->masks = reinterpret_cast<uint32_t*>(ws + L.masks);
    p->records = reinterpret_cast<uint4*>(ws + L.records);
    p->cls_cnt = reinterpret_cast<uint32_t*>(ws + L.cls_cnt);
    p->cls_flo = reinterpret_cast<uint32_t*>(ws + L.cls_flo);
    p->num_regions = (uint32_t)((p->num_points + kTile - 1) / kTile) * (kTile / kRegion);
    p->rec_cap = p->num_regions * (uint32_t)kRegion;
    p->rcnt = ws + L.rcnt;
    p->ckey = reinterpret_cast<unsigned long long*>(ws + L.ckey);
    p->key_b = reinterpret_cast<uint32_t*>(ws + L.ckey);
    p->val_b = p->key_b + (size_t)p->rec_cap;
    p->key_a = reinterpret_cast<uint32_t*>(ws + L.key_a);
    p->val_a = reinterpret_cast<uint32_t*>(ws + L.val_a);
    // pass k moves A to B for even k, B to A for odd k
    const bool in_b = (p->sort_passes & 1) != 0;
    p->skey = in_b ? p->key_b : p->key_a;
    p->sval = in_b ? p->val_b : p->val_a;
    p->fcnt = reinterpret_cast<uint32_t*>(ws + L.fcnt);
    p->ftot = reinterpret_cast<uint32_t*>(ws + L.ftot);
    p->hist = reinterpret_cast<uint32_t*>(ws + L.hist);
    p->sort_state = reinterpret_cast<unsigned long long*>(ws + L.sort_state);
    p->run_state = reinterpret_cast<unsigned long long*>(ws + L.run_state);
    // room for the look-back words of the radix passes and of the numbering
    p->sort_tiles_cap = L.sort_tiles_cap;
    p->run_tiles_cap = L.run_tiles_cap;
    p->vdesc = reinterpret_cast<uint4*>(ws + L.vdesc);
    p->mask_words = L.mask_words;
    p->coarse = L.coarse;
    p->coarse_inv[0] = (float)((double)L.coarse / ((double)p->rmax[0] - (double)p->rmin[0]));
    p->coarse_inv[1] = (float)((double)L.coarse / ((double)p->rmax[1] - (double)p->rmin[1]));
}

#define MMBEV_TRY(expr)                                   \
    do {                                                  \
        if ((expr) != cudaSuccess) return MMBEV_ECUDA;    \
    } while (0)

const char* const kStageNames[MMBEV_NUM_STAGES] = {
    "prep", "classify", "compact", "sort", "runs", "emit"};

}  // namespace

int num_sms() {
    static std::atomic<int> cache[64];
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) return 0;
    if (dev >= 0 && dev < 64) {
        const int c = cache[dev].load(std::memory_order_relaxed);
        if (c > 0) return c;
    }
    int n = 0;
    if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess) return 0;
    if (dev >= 0 && dev < 64) cache[dev].store(n, std::memory_order_relaxed);
    return n;
}

}  // namespace mmbev

using namespace mmbev;

extern "C" {

size_t mmbev_workspace_size(int64_t max_points, int32_t max_rois_per_frame, int32_t max_voxels,
                            int32_t num_frames, const float voxel_size[3], const float range[6]) {
    Grid g;
    if (max_points < 0 || max_points > kMaxPoints || max_rois_per_frame < 0 || max_rois_per_frame > kMaxRoisPerFrame ||
        max_voxels < 0 || num_frames < 1 || num_frames > kMaxFrames)
        return 0;
    if (!make_grid(voxel_size, range, &g)) return 0;
    const Layout L = make_layout(max_points, (int64_t)max_rois_per_frame * num_frames,
                                 max_rois_per_frame, max_voxels, num_frames, g);
    return L.total;
}

}  // extern "C"

namespace {

// The batched call; keep_status: leave the workspace's status word as it is
// (the chunks after the first of a host-input call).
int voxelize_batched(const float* points, const int64_t* sweep_offsets, int32_t num_sweeps,
                     const float* sweep_tf, const mmbev_roi_t* rois, int32_t num_rois,
                     float roi_margin, const float voxel_size[3], const float range[6],
                     int32_t max_pts_per_voxel, int32_t max_voxels, int32_t num_frames,
                     const int32_t* frame_sweep_offsets, const int32_t* frame_roi_offsets,
                     float* out_feats, int32_t* out_coords, int32_t* out_counts,
                     int32_t* out_nvox, void* workspace,
                     size_t workspace_bytes, cudaStream_t stream, const mmbev_exec_opts_t* opts,
                     bool keep_status) {
    HostDesc desc;  // ~25 KB; consumed by the prep launch's parameter copy
    Params p;
    Grid g;
    int32_t rmax = 0;
    if (max_pts_per_voxel < 1 || max_pts_per_voxel > kMaxK || max_voxels < 0) return MMBEV_EINVAL;
    if ((int64_t)max_voxels * num_frames > 0x7FFFFFFFll) return MMBEV_EINVAL;
    if (!out_nvox) return MMBEV_EINVAL;
    if (max_voxels > 0 && (!out_feats || !out_coords || !out_counts)) return MMBEV_EINVAL;
    if (!workspace || (reinterpret_cast<uintptr_t>(workspace) & (kAlign - 1))) return MMBEV_EINVAL;
    int rc = validate_common(points, sweep_offsets, num_sweeps, sweep_tf, rois, num_rois,
                             roi_margin, voxel_size, range, num_frames, frame_sweep_offsets,
                             frame_roi_offsets, &p, &desc, &g, &rmax);
    if (rc != MMBEV_OK) return rc;
    p.keep_status = keep_status ? 1 : 0;   // after validation, which resets p
    const Layout L = make_layout(p.num_points, num_rois, rmax, max_voxels, num_frames, g);
    if (L.total > workspace_bytes) return MMBEV_EWORKSPACE;
    bind_layout(&p, L, static_cast<uint8_t*>(workspace));
    p.K = max_pts_per_voxel;
    p.max_voxels = max_voxels;
    p.out_feats = out_feats;
    p.out_coords = out_coords;
    p.out_counts = out_counts;
    p.out_nvox = out_nvox;
    p.rho_thr = 0u;
    p.seed = 0ull;
    if (opts) {
        const float rho = opts->rho_out;
        if (!(rho >= 0.0f && rho <= 1.0f)) return MMBEV_EINVAL;
        // floor(rho * 2^24); rho = 1 keeps every draw
        p.rho_thr = rho >= 1.0f ? (1u << 24) : (uint32_t)std::floor((double)rho * 16777216.0);
        p.seed = opts->seed;
        p.inject_status = opts->inject_status;
    }

    const int sms = num_sms();
    if (sms <= 0) return MMBEV_ECUDA;
    {
        // classify: one block per SM (at most one per tile)
        const uint64_t tiles = ((uint64_t)p.num_points + kTile - 1) / kTile;
        uint64_t g = tiles < (uint64_t)sms ? tiles : (uint64_t)sms;
        if (g > (uint64_t)kMaxClsGrid) g = kMaxClsGrid;
        p.cls_grid = (uint32_t)g;
    }
    cudaEvent_t* ev = opts ? opts->stage_events : nullptr;
    int stage = 0;
    auto mark = [&]() -> cudaError_t {
        return ev ? cudaEventRecord(ev[stage++], stream) : cudaSuccess;
    };
    cudaError_t e = cudaSuccess;
    // The first kernel follows the stream's earlier work in full; the rest
    // are programmatic dependents of their predecessor (each waits for it
    // with griddepcontrol.wait before touching its results).
    const bool pdl = ev == nullptr;  // events between kernels break the chain anyway
    do {
        if ((e = mark()) != cudaSuccess) break;
        if ((e = launch_prep(p, desc, stream)) != cudaSuccess) break;
        if ((e = mark()) != cudaSuccess) break;
        if ((e = launch_classify(p, rmax, sms, pdl, stream)) != cudaSuccess) break;
        if ((e = mark()) != cudaSuccess) break;
        if ((e = launch_compact(p, sms, pdl, stream)) != cudaSuccess) break;
        if ((e = mark()) != cudaSuccess) break;
        if ((e = launch_sort(p, sms, pdl, stream)) != cudaSuccess) break;
        if ((e = mark()) != cudaSuccess) break;
        if ((e = launch_runs(p, sms, pdl, stream)) != cudaSuccess) break;
        if ((e = mark()) != cudaSuccess) break;
        if ((e = launch_emit(p, sms, pdl, stream)) != cudaSuccess) break;
        if ((e = mark()) != cudaSuccess) break;
    } while (0);
    return e == cudaSuccess ? MMBEV_OK : MMBEV_ECUDA;
}

}  // namespace

extern "C" {

int mmbev_voxelize_roi_batched_ex(const float* points, const int64_t* sweep_offsets,
                                  int32_t num_sweeps, const float* sweep_tf,
                                  const mmbev_roi_t* rois, int32_t num_rois, float roi_margin,
                                  const float voxel_size[3], const float range[6],
                                  int32_t max_pts_per_voxel, int32_t max_voxels,
                                  int32_t num_frames, const int32_t* frame_sweep_offsets,
                                  const int32_t* frame_roi_offsets, float* out_feats,
                                  int32_t* out_coords, int32_t* out_counts, int32_t* out_nvox,
                                  void* workspace,
                                  size_t workspace_bytes, cudaStream_t stream,
                                  const mmbev_exec_opts_t* opts) {
    return voxelize_batched(points, sweep_offsets, num_sweeps, sweep_tf, rois, num_rois,
                            roi_margin, voxel_size, range, max_pts_per_voxel, max_voxels,
                            num_frames, frame_sweep_offsets, frame_roi_offsets, out_feats,
                            out_coords, out_counts, out_nvox, workspace,
                            workspace_bytes, stream, opts, false);
}

int mmbev_voxelize_roi_batched_host(
    const float* h_points, const int64_t* sweep_offsets, int32_t num_sweeps,
    const float* h_sweep_tf, const mmbev_roi_t* h_rois, int32_t num_rois, float roi_margin,
    const float voxel_size[3], const float range[6], int32_t max_pts_per_voxel,
    int32_t max_voxels, int32_t num_frames, const int32_t* frame_sweep_offsets,
    const int32_t* frame_roi_offsets, float* d_points, float* d_sweep_tf, mmbev_roi_t* d_rois,
    float* out_feats, int32_t* out_coords, int32_t* out_counts, int32_t* out_nvox,
    void* workspace, size_t workspace_bytes, void* pack_dst,
    size_t pack_bytes, int32_t chunk_frames, cudaStream_t stream, cudaStream_t copy_stream,
    const mmbev_exec_opts_t* opts) {
    if (num_frames < 1 || num_frames > kMaxFrames || chunk_frames < 1) return MMBEV_EINVAL;
    if (num_sweeps < 0 || num_sweeps > kMaxSweeps || num_rois < 0) return MMBEV_EINVAL;
    if (!out_nvox) return MMBEV_EINVAL;
    if (!sweep_offsets || !frame_sweep_offsets || !frame_roi_offsets) return MMBEV_EINVAL;
    if (opts && opts->stage_events) return MMBEV_EINVAL;   // stage events need a single call
    if (max_voxels < 0 || (int64_t)max_voxels * num_frames > 0x7FFFFFFFll) return MMBEV_EINVAL;
    // the offsets this entry slices by: checked before any copy
    if (frame_sweep_offsets[0] != 0 || frame_sweep_offsets[num_frames] != num_sweeps ||
        frame_roi_offsets[0] != 0 || frame_roi_offsets[num_frames] != num_rois ||
        sweep_offsets[0] != 0)
        return MMBEV_EINVAL;
    for (int32_t f = 0; f < num_frames; ++f)
        if (frame_sweep_offsets[f + 1] < frame_sweep_offsets[f] ||
            frame_roi_offsets[f + 1] < frame_roi_offsets[f])
            return MMBEV_EINVAL;
    for (int32_t s = 0; s < num_sweeps; ++s)
        if (sweep_offsets[s + 1] < sweep_offsets[s]) return MMBEV_EINVAL;
    if (pack_dst && ((reinterpret_cast<uintptr_t>(pack_dst) & 3u) || max_voxels == 0))
        return MMBEV_EINVAL;
    if (pack_dst && pack_bytes < mmbev_pack_size(num_frames, max_voxels)) return MMBEV_EWORKSPACE;
    const int64_t n = sweep_offsets[num_sweeps];
    if ((n > 0 && (!h_points || !d_points)) || (num_sweeps > 0 && (!h_sweep_tf || !d_sweep_tf)) ||
        (num_rois > 0 && (!h_rois || !d_rois)))
        return MMBEV_EINVAL;

    const int32_t nchunks = (num_frames + chunk_frames - 1) / chunk_frames;
    std::vector<cudaEvent_t> ev((size_t)nchunks, nullptr);
    std::vector<int64_t> so;
    std::vector<int32_t> fso, fro;
    int rc = MMBEV_OK;
    for (int32_t c = 0; c < nchunks && rc == MMBEV_OK; ++c) {
        const int32_t f0 = c * chunk_frames, f1 = std::min(num_frames, f0 + chunk_frames);
        const int32_t s0 = frame_sweep_offsets[f0], s1 = frame_sweep_offsets[f1];
        const int32_t r0 = frame_roi_offsets[f0], r1 = frame_roi_offsets[f1];
        const int64_t p0 = sweep_offsets[s0], p1 = sweep_offsets[s1];
        // the chunk's inputs go up on the copy stream; the compute stream
        // waits for them only
        cudaError_t e = cudaEventCreateWithFlags(&ev[(size_t)c], cudaEventDisableTiming);
        if (e == cudaSuccess && p1 > p0)
            e = cudaMemcpyAsync(d_points + 5 * p0, h_points + 5 * p0,
                                sizeof(float) * 5 * (size_t)(p1 - p0), cudaMemcpyHostToDevice,
                                copy_stream);
        if (e == cudaSuccess && s1 > s0)
            e = cudaMemcpyAsync(d_sweep_tf + 16 * (size_t)s0, h_sweep_tf + 16 * (size_t)s0,
                                sizeof(float) * 16 * (size_t)(s1 - s0), cudaMemcpyHostToDevice,
                                copy_stream);
        if (e == cudaSuccess && r1 > r0)
            e = cudaMemcpyAsync(d_rois + r0, h_rois + r0, sizeof(mmbev_roi_t) * (size_t)(r1 - r0),
                                cudaMemcpyHostToDevice, copy_stream);
        if (e == cudaSuccess) e = cudaEventRecord(ev[(size_t)c], copy_stream);
        if (e == cudaSuccess) e = cudaStreamWaitEvent(stream, ev[(size_t)c], 0);
        if (e != cudaSuccess) {
            rc = MMBEV_ECUDA;
            break;
        }
        // the chunk's offsets, rebased (taken by value at launch)
        so.assign(sweep_offsets + s0, sweep_offsets + s1 + 1);
        for (int64_t& v : so) v -= p0;
        fso.assign(frame_sweep_offsets + f0, frame_sweep_offsets + f1 + 1);
        for (int32_t& v : fso) v -= s0;
        fro.assign(frame_roi_offsets + f0, frame_roi_offsets + f1 + 1);
        for (int32_t& v : fro) v -= r0;
        const size_t row0 = (size_t)f0 * (size_t)max_voxels;
        // a test hook's status bits go into the first chunk only
        mmbev_exec_opts_t copts{};
        if (opts) {
            copts = *opts;
            if (c > 0) copts.inject_status = 0u;
        }
        rc = voxelize_batched(
            d_points ? d_points + 5 * p0 : nullptr, so.data(), s1 - s0,
            d_sweep_tf ? d_sweep_tf + 16 * (size_t)s0 : nullptr, d_rois ? d_rois + r0 : nullptr,
            r1 - r0, roi_margin, voxel_size, range, max_pts_per_voxel, max_voxels, f1 - f0,
            fso.data(), fro.data(), out_feats ? out_feats + 5 * row0 : nullptr,
            out_coords ? out_coords + 3 * row0 : nullptr,
            out_counts ? out_counts + row0 : nullptr, out_nvox + f0,
            workspace, workspace_bytes, stream, opts ? &copts : nullptr, c > 0);
        // the chunk's kept rows into the packed buffer (offsets of frames
        // f0..f1 and their records), while later chunks go up and run
        if (rc == MMBEV_OK && pack_dst &&
            launch_pack(out_feats, out_coords, out_counts, out_nvox, num_frames, f0, f1,
                        max_voxels, pack_dst, stream) != cudaSuccess)
            rc = MMBEV_ECUDA;
    }
    for (cudaEvent_t x : ev)
        if (x) cudaEventDestroy(x);   // released once the work recorded on it is done
    return rc;
}

int mmbev_voxelize_roi_batched(const float* points, const int64_t* sweep_offsets,
                               int32_t num_sweeps, const float* sweep_tf,
                               const mmbev_roi_t* rois, int32_t num_rois, float roi_margin,
                               const float voxel_size[3], const float range[6],
                               int32_t max_pts_per_voxel, int32_t max_voxels, int32_t num_frames,
                               const int32_t* frame_sweep_offsets,
                               const int32_t* frame_roi_offsets, float* out_feats,
                               int32_t* out_coords, int32_t* out_counts, int32_t* out_nvox,
                               void* workspace,
                               size_t workspace_bytes, cudaStream_t stream) {
    return mmbev_voxelize_roi_batched_ex(points, sweep_offsets, num_sweeps, sweep_tf, rois,
                                         num_rois, roi_margin, voxel_size, range,
                                         max_pts_per_voxel, max_voxels, num_frames,
                                         frame_sweep_offsets, frame_roi_offsets, out_feats,
                                         out_coords, out_counts, out_nvox,
                                         workspace, workspace_bytes, stream, nullptr);
}

int mmbev_voxelize_roi(const float* points, const int64_t* sweep_offsets, int32_t num_sweeps,
                       const float* sweep_tf, const mmbev_roi_t* rois, int32_t num_rois,
                       float roi_margin, const float voxel_size[3], const float range[6],
                       int32_t max_pts_per_voxel, int32_t max_voxels, float* out_feats,
                       int32_t* out_coords, int32_t* out_counts, int32_t* out_nvox,
                       void* workspace, size_t workspace_bytes,
                       cudaStream_t stream) {
    const int32_t fso[2] = {0, num_sweeps};
    const int32_t fro[2] = {0, num_rois};
    return mmbev_voxelize_roi_batched_ex(points, sweep_offsets, num_sweeps, sweep_tf, rois,
                                         num_rois, roi_margin, voxel_size, range,
                                         max_pts_per_voxel, max_voxels, 1, fso, fro, out_feats,
                                         out_coords, out_counts, out_nvox,
                                         workspace, workspace_bytes, stream, nullptr);
}

int mmbev_classify_points(const float* points, const int64_t* sweep_offsets, int32_t num_sweeps,
                          const float* sweep_tf, const mmbev_roi_t* rois, int32_t num_rois,
                          float roi_margin, const float voxel_size[3], const float range[6],
                          int32_t num_frames, const int32_t* frame_sweep_offsets,
                          const int32_t* frame_roi_offsets, float* out_xyz, int64_t* out_lin,
                          int32_t* out_rank, void* workspace, size_t workspace_bytes,
                          cudaStream_t stream) {
    HostDesc desc;
    Params p;
    Grid g;
    int32_t rmax = 0;
    if (!workspace || (reinterpret_cast<uintptr_t>(workspace) & (kAlign - 1))) return MMBEV_EINVAL;
    int rc = validate_common(points, sweep_offsets, num_sweeps, sweep_tf, rois, num_rois,
                             roi_margin, voxel_size, range, num_frames, frame_sweep_offsets,
                             frame_roi_offsets, &p, &desc, &g, &rmax);
    if (rc == MMBEV_OK && p.num_points > 0 && (!out_xyz || !out_lin || !out_rank)) rc = MMBEV_EINVAL;
    if (rc != MMBEV_OK) return rc;
    const Layout L = make_layout(p.num_points, num_rois, rmax, 0, num_frames, g);
    if (L.total > workspace_bytes) return MMBEV_EWORKSPACE;
    bind_layout(&p, L, static_cast<uint8_t*>(workspace));
    p.K = 1;
    p.cls_xyz = out_xyz;
    p.cls_lin = out_lin;
    p.cls_rank = out_rank;
    cudaError_t e = launch_prep(p, desc, stream);
    if (e == cudaSuccess) e = launch_classify_points(p, stream);
    return e == cudaSuccess ? MMBEV_OK : MMBEV_ECUDA;
}

int mmbev_prep_rois(const mmbev_roi_t* rois, int32_t num_rois, float roi_margin, float* out,
                    cudaStream_t stream) {
    if (num_rois < 0 || (num_rois > 0 && (!rois || !out))) return MMBEV_EINVAL;
    if (!std::isfinite(roi_margin) || !(roi_margin >= 0.0f)) return MMBEV_EINVAL;
    return launch_prep_rois(rois, num_rois, roi_margin, out, stream) == cudaSuccess ? MMBEV_OK
                                                                                   : MMBEV_ECUDA;
}

int mmbev_get_status(const void* workspace, size_t workspace_bytes, uint32_t* host_status,
                     cudaStream_t stream) {
    if (!workspace || !host_status || workspace_bytes < sizeof(Header)) return MMBEV_EINVAL;
    const Header* hdr = static_cast<const Header*>(workspace);
    MMBEV_TRY(cudaMemcpyAsync(host_status, &hdr->status, sizeof(uint32_t),
                              cudaMemcpyDeviceToHost, stream));
    MMBEV_TRY(cudaStreamSynchronize(stream));
    return MMBEV_OK;
}

const char* mmbev_stage_name(int32_t stage) {
    if (stage < 0 || stage >= MMBEV_NUM_STAGES) return "";
    return kStageNames[stage];
}

const char* mmbev_version(void) { return "mmbev 0.1.0 (sm_103a)"; }

}  // extern "C"
