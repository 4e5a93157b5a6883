// Packing of a voxelize call's kept rows: every frame's rows [0, nvox[f])
// gathered, frame after frame, into one contiguous buffer. The caller copies
// it in one transfer, or passes pinned host memory and the device writes it
// there directly over the host link.
//
// Layout of dst: int32 off[F+1] (off[f] = the first record of frame f,
// off[F] = the total T), then T records of nine 4-byte words: the five fp32
// means, then z, y, x and the point count as int32.
//
// One kernel: every block scans nvox into shared memory (F <= 1024 frames),
// then each warp takes 32 consecutive records at a time: a lane finds its
// record's frame by binary search, and the warp writes the 288 words of the
// 32 records as nine stores of 32 consecutive words. A launch may cover a
// range of frames [f0, f1): it writes off[f0..f1] and those frames' records,
// so a batch can be packed chunk by chunk as its chunks complete.
#include <cstdint>

#include "mmbev_internal.cuh"

namespace mmbev {
namespace {

constexpr int kPackThreads = 256;
constexpr int kPackPer = (kMaxFrames + kPackThreads - 1) / kPackThreads;   // frames a thread scans

__global__ void __launch_bounds__(kPackThreads)
k_pack(const float* __restrict__ feats, const int32_t* __restrict__ coords,
       const int32_t* __restrict__ counts, const int32_t* __restrict__ nvox, int32_t F,
       int32_t f0, int32_t f1, int32_t max_voxels, int32_t* dst) {
    __shared__ int32_t s_off[kMaxFrames + 1];
    __shared__ int32_t s_warp[kPackThreads / 32];
    const int t = threadIdx.x, lane = t & 31, wid = t >> 5;

    // exclusive prefix of min(max(nvox[f], 0), max_voxels) over frames
    // [0, f1): kPackPer frames a thread, then a scan across the block
    int32_t mine[kPackPer];
    int32_t sum = 0;
#pragma unroll
    for (int i = 0; i < kPackPer; ++i) {
        const int f = t * kPackPer + i;
        mine[i] = f < f1 ? min(max(__ldg(nvox + f), 0), max_voxels) : 0;
        sum += mine[i];
    }
    int32_t incl = sum;
#pragma unroll
    for (int d = 1; d < 32; d <<= 1) {
        const int32_t o = __shfl_up_sync(0xFFFFFFFFu, incl, d);
        if (lane >= d) incl += o;
    }
    if (lane == 31) s_warp[wid] = incl;
    __syncthreads();
    int32_t before = incl - sum;
    for (int w = 0; w < wid; ++w) before += s_warp[w];
#pragma unroll
    for (int i = 0; i < kPackPer; ++i) {
        const int f = t * kPackPer + i;
        if (f < f1) s_off[f] = before;
        before += mine[i];
    }
    if (t == kPackThreads - 1) s_off[f1] = before;   // the last thread's running sum
    __syncthreads();
    const int32_t T = s_off[f1];   // records before frame f1
    if (blockIdx.x == 0)
        for (int f = f0 + t; f <= f1; f += kPackThreads) dst[f] = s_off[f];

    uint32_t* rec = reinterpret_cast<uint32_t*>(dst + F + 1);
    const size_t nwarps = (size_t)gridDim.x * (kPackThreads / 32);
    const size_t first = (size_t)s_off[f0];   // this range's records: [first, T)
    for (size_t p0 = first + ((size_t)blockIdx.x * (kPackThreads / 32) + wid) * 32; p0 < (size_t)T;
         p0 += nwarps * 32) {
        const size_t p = p0 + lane;
        unsigned long long src = 0;
        if (p < (size_t)T) {
            int lo = f0, hi = f1;   // the last f with s_off[f] <= p
            while (hi - lo > 1) {
                const int mid = (lo + hi) >> 1;
                if ((size_t)s_off[mid] <= p) lo = mid;
                else hi = mid;
            }
            src = (unsigned long long)lo * (unsigned long long)max_voxels + (p - (size_t)s_off[lo]);
        }
        const int nrec = (int)min((size_t)32, (size_t)T - p0);
        uint32_t* out = rec + p0 * 9;   // record p0 of the whole batch
#pragma unroll
        for (int k = 0; k < 9; ++k) {
            const int w = k * 32 + lane;   // word of the warp's block of 32 records
            const int r = w / 9, c = w - 9 * (w / 9);
            const unsigned long long s = __shfl_sync(0xFFFFFFFFu, src, r);
            if (r < nrec) {
                const uint32_t val =
                    c < 5 ? __float_as_uint(__ldg(feats + 5 * s + c))
                          : (uint32_t)(c < 8 ? __ldg(coords + 3 * s + (c - 5)) : __ldg(counts + s));
                out[w] = val;
            }
        }
    }
}

}  // namespace

cudaError_t launch_pack(const float* feats, const int32_t* coords, const int32_t* counts,
                        const int32_t* nvox, int32_t F, int32_t f0, int32_t f1,
                        int32_t max_voxels, void* dst, cudaStream_t stream) {
    const int sms = num_sms();
    if (sms <= 0) return cudaErrorInvalidDevice;
    k_pack<<<(unsigned)sms * 2, kPackThreads, 0, stream>>>(feats, coords, counts, nvox, F, f0, f1,
                                                            max_voxels,
                                                            static_cast<int32_t*>(dst));
    return cudaGetLastError();
}

}  // namespace mmbev

using namespace mmbev;

extern "C" size_t mmbev_pack_size(int32_t num_frames, int32_t max_voxels) {
    if (num_frames < 0 || num_frames > kMaxFrames || max_voxels < 0) return 0;
    return sizeof(int32_t) * ((size_t)num_frames + 1) +
           36u * (size_t)num_frames * (size_t)max_voxels;
}

extern "C" int mmbev_pack_voxels(const float* feats, const int32_t* coords, const int32_t* counts,
                                 const int32_t* nvox, int32_t num_frames, int32_t max_voxels,
                                 void* dst, size_t dst_bytes, cudaStream_t stream) {
    if (num_frames < 0 || num_frames > kMaxFrames || max_voxels < 0) return MMBEV_EINVAL;
    if ((unsigned long long)num_frames * (unsigned long long)max_voxels > 0x7FFFFFFFull)
        return MMBEV_EINVAL;
    if (!dst || (reinterpret_cast<uintptr_t>(dst) & 3u)) return MMBEV_EINVAL;
    if (dst_bytes < mmbev_pack_size(num_frames, max_voxels)) return MMBEV_EWORKSPACE;
    if (num_frames > 0 && (!feats || !coords || !counts || !nvox)) return MMBEV_EINVAL;
    return launch_pack(feats, coords, counts, nvox, num_frames, 0, num_frames, max_voxels, dst,
                       stream) == cudaSuccess
               ? MMBEV_OK
               : MMBEV_ECUDA;
}
