// Question-time snapshot / restore of a stream's state (Sec. 3.3, "Question answering"): a batch
// of row copies in one launch.
//
// The bytes move at HBM bandwidth with nothing to compute, so the kernel is a plain streaming
// copy: each segment's rows form one index space of 16-byte vectors, walked grid-stride with four
// independent loads in flight per thread (evict-first: the copy is not read again soon), and the
// grid is a few CTAs per SM so that about 64 KB per SM is in flight, enough to cover the DRAM
// latency.
#include <algorithm>

#include "internal.cuh"

namespace deltas {
namespace {

constexpr int kCopyThreads = 256;
constexpr int kCopyCtasPerSm = 4;

__global__ void __launch_bounds__(kCopyThreads)
copy_batch_kernel(const __grid_constant__ CopyBatch b)
{
    const uint64_t nth = (uint64_t)gridDim.x * kCopyThreads;
    const uint64_t t0 = (uint64_t)blockIdx.x * kCopyThreads + threadIdx.x;
    for (int s = 0; s < b.n; ++s) {
        const CopySeg g = b.seg[s];
        const uint64_t nv = g.row_bytes >> 4;              // whole 16-byte vectors per row
        const uint64_t nw = (g.row_bytes & 15) >> 2;       // then 4-byte words
        // the segment's rows as one index space of vectors, so that every thread keeps four
        // loads in flight however short the rows are; thread t copies vectors t + k nth
        // (k = 0, 1, 2, 3), then each of the four moves on by 4 nth: four (row, column) cursors,
        // advanced without a division
        const uint64_t total = nv * (uint64_t)g.rows;
        if (total > 0) {
            const uint64_t step = 4 * nth, q = step / nv, m = step - q * nv;
            uint64_t cr[4], cc[4];
#pragma unroll
            for (int k = 0; k < 4; ++k) {
                const uint64_t v = t0 + k * nth;
                cr[k] = v / nv;
                cc[k] = v - cr[k] * nv;
            }
            auto src_at = [&](int k) {
                return reinterpret_cast<const uint4*>(g.src + cr[k] * g.stride) + cc[k];
            };
            auto dst_at = [&](int k) { return reinterpret_cast<uint4*>(g.dst + cr[k] * g.stride) + cc[k]; };
            uint64_t v = t0;
            for (; v + 3 * nth < total; v += step) {
                uint4 x[4];
#pragma unroll
                for (int k = 0; k < 4; ++k) x[k] = __ldcs(src_at(k));
#pragma unroll
                for (int k = 0; k < 4; ++k) __stcs(dst_at(k), x[k]);
#pragma unroll
                for (int k = 0; k < 4; ++k) {
                    cc[k] += m;
                    cr[k] += q;
                    if (cc[k] >= nv) { cc[k] -= nv; ++cr[k]; }
                }
            }
#pragma unroll
            for (int k = 0; k < 3; ++k)
                if (v + k * nth < total) __stcs(dst_at(k), __ldcs(src_at(k)));
        }
        // rows whose length is not a multiple of 16 bytes: their last 4-byte words
        for (uint64_t w = t0; w < nw * (uint64_t)g.rows; w += nth) {
            const uint64_t r = w / nw, c = w - r * nw;
            reinterpret_cast<uint32_t*>(g.dst + r * g.stride + nv * 16)[c] =
                reinterpret_cast<const uint32_t*>(g.src + r * g.stride + nv * 16)[c];
        }
    }
}

}  // namespace

cudaError_t launch_copy_batch(const CopyBatch& b, cudaStream_t s)
{
    uint64_t vec = 0;
    for (int i = 0; i < b.n; ++i) vec += (b.seg[i].row_bytes >> 4) * (uint64_t)b.seg[i].rows;
    if (b.n == 0) return cudaSuccess;
    // enough threads for four vectors each, at most kCopyCtasPerSm CTAs per SM
    const uint64_t want = (vec + 4ull * kCopyThreads - 1) / (4ull * kCopyThreads);
    const int grid = (int)std::max<uint64_t>(1, std::min<uint64_t>(want, (uint64_t)device_sm_count() * kCopyCtasPerSm));
    copy_batch_kernel<<<grid, kCopyThreads, 0, s>>>(b);
    return cudaGetLastError();
}

}  // namespace deltas
