// State drift (Sec. 3.2, Eq. 3) from two stored states, and the chunk score from drift partials.
//
// state_drift: one CTA per (layer, value head) streams both d_v x d_k states once with 16-byte
// loads, four pairs in flight per thread (HBM-bound: 2 * 4 * d_v * d_k bytes per head), and writes
//   partials[l][h] = { sum (S_after - S_before)^2, sum S_before^2 }.
// The difference is formed element by element before squaring, never as
// |A|^2 - 2<A,B> + |B|^2, which cancels badly when the drift is small.
//
// score_chunks: one CTA reduces the [L][Hv][2] partials in a fixed order (one warp per layer:
// lane-strided float sums over the heads, a fixed xor tree), applies sqrt(num_l)/sqrt(den_l) per
// layer in float with the zero-norm reading (0/0 -> 0, x/0 -> +inf), adds the layer terms in
// double in a fixed order and stores the layer mean as the chunk's score.
#include "internal.cuh"

namespace deltas {
namespace {

constexpr int kDriftThreads = 256;
constexpr int kDriftUnroll = 4;        // float4 pairs in flight per thread

__global__ void __launch_bounds__(kDriftThreads)
state_drift_kernel(int n_elem4, const float4* __restrict__ sb, const float4* __restrict__ sa,
                   float* __restrict__ partials)
{
    const size_t base = (size_t)blockIdx.x * n_elem4;
    float num = 0.f, den = 0.f;
    for (int e = threadIdx.x; e < n_elem4; e += kDriftThreads * kDriftUnroll) {
        float4 b[kDriftUnroll], a[kDriftUnroll];
#pragma unroll
        for (int u = 0; u < kDriftUnroll; ++u) {          // every load issued before any use
            const int i = e + u * kDriftThreads;
            if (i < n_elem4) { b[u] = __ldcs(sb + base + i); a[u] = __ldcs(sa + base + i); }   // streamed once
            else { b[u] = make_float4(0.f, 0.f, 0.f, 0.f); a[u] = b[u]; }
        }
#pragma unroll
        for (int u = 0; u < kDriftUnroll; ++u) {
            const float dx = a[u].x - b[u].x, dy = a[u].y - b[u].y, dz = a[u].z - b[u].z, dw = a[u].w - b[u].w;
            num += dx * dx + dy * dy + dz * dz + dw * dw;
            den += b[u].x * b[u].x + b[u].y * b[u].y + b[u].z * b[u].z + b[u].w * b[u].w;
        }
    }
    // a pairwise tree over the warp in float (the FP64 pipe is slow on this part), then the
    // warps' sums added in double in warp order
#pragma unroll
    for (int m = 16; m >= 1; m >>= 1) {
        num += __shfl_xor_sync(0xffffffffu, num, m);
        den += __shfl_xor_sync(0xffffffffu, den, m);
    }
    const double dn = num, dd = den;
    __shared__ double red[2][kDriftThreads / 32];
    if ((threadIdx.x & 31) == 0) { red[0][threadIdx.x >> 5] = dn; red[1][threadIdx.x >> 5] = dd; }
    __syncthreads();
    if (threadIdx.x == 0) {
        double sn = 0.0, sd = 0.0;
        for (int w = 0; w < kDriftThreads / 32; ++w) { sn += red[0][w]; sd += red[1][w]; }
        partials[(size_t)blockIdx.x * 2 + 0] = (float)sn;
        partials[(size_t)blockIdx.x * 2 + 1] = (float)sd;
    }
}

constexpr int kScoreThreads = 1024;

// One warp per layer (layers strided over the 32 warps): lane-strided float sums over the heads and
// a fixed xor tree (pairwise: a few ulp of float), the layer's ratio in float on lane 0, then
// warp 0 adds the layer terms in layer order in double.  (The FP64 pipe is slow on this part, so
// double arithmetic is kept to one addition per layer.)
__global__ void __launch_bounds__(kScoreThreads)
score_chunks_kernel(int L, int Hv, const float* __restrict__ partials, int chunk_id,
                    float* __restrict__ scores)
{
    __shared__ double term_sum[kScoreThreads / 32];
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    grid_dep_launch();                                 // the next call's kernel may be scheduled now
    grid_dep_wait();                                   // the partials are written
    double acc = 0.0;
    for (int l = warp; l < L; l += kScoreThreads / 32) {
        float num = 0.f, den = 0.f;
        for (int h = lane; h < Hv; h += 32) {
            num += partials[((size_t)l * Hv + h) * 2 + 0];
            den += partials[((size_t)l * Hv + h) * 2 + 1];
        }
#pragma unroll
        for (int m = 16; m >= 1; m >>= 1) {
            num += __shfl_xor_sync(0xffffffffu, num, m);
            den += __shfl_xor_sync(0xffffffffu, den, m);
        }
        if (lane == 0) {
            double term;
            if (den > 0.f) term = (double)(sqrtf(num) / sqrtf(den));
            else term = (num > 0.f) ? (double)INFINITY : 0.0;
            acc += term;   // layers l, l + 32, ... in increasing order
        }
    }
    if (lane == 0) term_sum[warp] = acc;
    __syncthreads();
    if (threadIdx.x == 0) {
        double total = 0.0;
        for (int w = 0; w < kScoreThreads / 32; ++w) total += term_sum[w];
        scores[chunk_id] = (float)(total / (double)L);
    }
}

// The comparison signal's chunk score (Sec. 4.3): write sizes averaged over the heads, the layers
// and the chunk's tokens, i.e. their total over L * Hv * n_tokens; the total is summed in double
// in a fixed order (one warp, lane-strided, then a fixed xor tree).
__global__ void __launch_bounds__(32)
score_write_norms_kernel(int n, const float* __restrict__ wnorm, double inv_count, int chunk_id,
                         float* __restrict__ scores)
{
    grid_dep_launch();                                 // the next call's kernel may be scheduled now
    grid_dep_wait();                                   // the write sizes are written
    double acc = 0.0;
    for (int i = threadIdx.x; i < n; i += 32) acc += (double)wnorm[i];
#pragma unroll
    for (int m = 16; m >= 1; m >>= 1) acc += __shfl_xor_sync(0xffffffffu, acc, m);
    if (threadIdx.x == 0) scores[chunk_id] = (float)(acc * inv_count);
}

}  // namespace

cudaError_t launch_score_write_norms(int L, int Hv, const float* wnorm, int n_tokens, int chunk_id, float* scores,
                                     cudaStream_t s)
{
    const double inv = n_tokens > 0 ? 1.0 / ((double)L * Hv * n_tokens) : 0.0;
    // scheduled while the update finishes (it waits for it before reading)
    return launch_dependent(score_write_norms_kernel, dim3(1), dim3(32), 0, s, L * Hv, wnorm, inv, chunk_id, scores);
}

cudaError_t launch_state_drift(int L, int Hv, int dv, int dk, const float* sb, const float* sa,
                               float* partials, cudaStream_t s)
{
    const int n4 = dv * dk / 4;
    state_drift_kernel<<<L * Hv, kDriftThreads, 0, s>>>(n4, reinterpret_cast<const float4*>(sb),
                                                        reinterpret_cast<const float4*>(sa), partials);
    return cudaGetLastError();
}

cudaError_t launch_score_chunks(int L, int Hv, const float* partials, int chunk_id, float* scores,
                                cudaStream_t s)
{
    // scheduled while the update finishes (it waits for it before reading)
    return launch_dependent(score_chunks_kernel, dim3(1), dim3(kScoreThreads), 0, s, L, Hv, partials, chunk_id,
                            scores);
}

}  // namespace deltas
