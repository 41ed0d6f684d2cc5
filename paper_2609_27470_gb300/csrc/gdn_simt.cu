// Gated delta rule over one chunk on CUDA cores, token by token, with the drift partials fused.
//
// Paper: Sec. 3.2, Eq. 2  S_t = alpha_t S_{t-1} + beta_t (v_t - alpha_t S_{t-1} k_t) k_t^T,
// Eq. 3 numerator/denominator per (layer, head).  This is the general-shape kernel (any
// d in {16, 32, 64, 128}, float32 or bfloat16 activations); the tensor-core kernel in
// gdn_tc.cu takes the d = 128 bfloat16 case.
//
// One CTA owns one (layer, value head).  Its d_v x d_k state lives in registers for the whole
// chunk: thread (row, sub) holds row `row`, float4 column groups sub, sub + TPR, ... (interleaved
// so that the TPR threads of a row read the staged key with distinct shared-memory banks).  Per
// token: r = S k (TPR-lane shuffle reduction), u = beta (v - alpha r), S = alpha S + u k^T.  The
// state before the chunk stays in registers too, so the drift partials need no second read of
// the state from memory.  Optionally the same pass sums the write sizes ||u_t|| (u = beta (v -
// alpha r), the comparison signal of Sec. 4.3) over the chunk: each warp adds its rows' u^2 for
// the token into shared memory, and after each staged pass one thread takes the square roots.
#include "internal.cuh"

namespace deltas {
namespace {

template <int D> struct SimtShape {
    static constexpr int TPR = D >= 32 ? D / 32 : 1;   // threads per state row
    static constexpr int SEG = D / TPR;                // columns per thread
    static constexpr int NG = SEG / 4;                 // float4 groups per thread
    static constexpr int NT = D * TPR;                 // threads per CTA
    static constexpr int TB = D >= 128 ? 16 : 32;      // tokens staged per pass
};

template <typename Tin, int D>
__global__ void __launch_bounds__(SimtShape<D>::NT)
gdn_update_simt_kernel(GdnArgs a)
{
    using Sh = SimtShape<D>;
    constexpr int TPR = Sh::TPR, NG = Sh::NG, NT = Sh::NT, TB = Sh::TB;
    __shared__ __align__(16) float sk[TB][D];
    __shared__ __align__(16) float sq[TB][D];
    __shared__ __align__(16) float sv[TB][D];
    __shared__ __align__(16) float so[TB][D];
    __shared__ float salpha[TB], sbeta[TB];
    __shared__ float su2[TB];                        // per-token sum of u^2 over the rows
    __shared__ double red[2][NT / 32 + 1];

    const int lh = blockIdx.x;
    const int l = lh / a.Hv, h = lh % a.Hv;
    const int kh = (int)(((long long)h * a.Hk) / a.Hv);
    const int tid = threadIdx.x;
    const int row = tid / TPR, sub = tid % TPR;
    const bool want_out = a.out != nullptr;
    const bool want_w = a.wnorm != nullptr;
    constexpr unsigned kLanes = NT >= 32 ? 0xffffffffu : ((1u << NT) - 1u);
    float wsum = 0.f;                                // thread 0: sum over tokens of ||u_t||
    for (int e = tid; e < TB; e += NT) su2[e] = 0.f;

    float* Srow = a.state + ((size_t)lh * D + row) * D;
    float4 S[NG], S0[NG];
#pragma unroll
    for (int j = 0; j < NG; ++j) {
        S[j] = *reinterpret_cast<const float4*>(Srow + 4 * (j * TPR + sub));
        S0[j] = S[j];
    }

    const Tin* kin = static_cast<const Tin*>(a.k);
    const Tin* qin = static_cast<const Tin*>(a.q);
    const Tin* vin = static_cast<const Tin*>(a.v);
    Tin* oout = static_cast<Tin*>(a.out);

    for (int t0 = 0; t0 < a.T; t0 += TB) {
        const int nt = min(TB, a.T - t0);
        __syncthreads();
        for (int e = tid; e < nt * D; e += NT) {
            const int tt = e / D, c = e % D;
            const size_t tok = (size_t)l * a.T + t0 + tt;
            sk[tt][c] = to_f32(kin[(tok * a.Hk + kh) * D + c]);
            sv[tt][c] = to_f32(vin[(tok * a.Hv + h) * D + c]);
            if (want_out) sq[tt][c] = to_f32(qin[(tok * a.Hk + kh) * D + c]);
        }
        for (int e = tid; e < nt; e += NT) {
            const size_t gi = ((size_t)l * a.T + t0 + e) * a.Hv + h;
            salpha[e] = expf(a.g[gi]);
            sbeta[e] = a.beta[gi];
        }
        __syncthreads();
        for (int tt = 0; tt < nt; ++tt) {
            const float4* kv4 = reinterpret_cast<const float4*>(sk[tt]);
            float r = 0.f;
#pragma unroll
            for (int j = 0; j < NG; ++j) {
                const float4 kk = kv4[j * TPR + sub];
                r = fmaf(S[j].x, kk.x, r);
                r = fmaf(S[j].y, kk.y, r);
                r = fmaf(S[j].z, kk.z, r);
                r = fmaf(S[j].w, kk.w, r);
            }
#pragma unroll
            for (int m = 1; m < TPR; m <<= 1) r += __shfl_xor_sync(0xffffffffu, r, m);
            const float alpha = salpha[tt];
            const float u = sbeta[tt] * (sv[tt][row] - alpha * r);
            if (want_w) {
                float u2 = sub == 0 ? u * u : 0.f;          // the TPR threads of a row share u
#pragma unroll
                for (int m = (NT >= 32 ? 16 : NT / 2); m >= 1; m >>= 1) u2 += __shfl_xor_sync(kLanes, u2, m);
                if ((tid & 31) == 0) atomicAdd(&su2[tt], u2);
            }
#pragma unroll
            for (int j = 0; j < NG; ++j) {
                const float4 kk = kv4[j * TPR + sub];
                S[j].x = fmaf(u, kk.x, alpha * S[j].x);
                S[j].y = fmaf(u, kk.y, alpha * S[j].y);
                S[j].z = fmaf(u, kk.z, alpha * S[j].z);
                S[j].w = fmaf(u, kk.w, alpha * S[j].w);
            }
            if (want_out) {
                const float4* qv4 = reinterpret_cast<const float4*>(sq[tt]);
                float o = 0.f;
#pragma unroll
                for (int j = 0; j < NG; ++j) {
                    const float4 qq = qv4[j * TPR + sub];
                    o = fmaf(S[j].x, qq.x, o);
                    o = fmaf(S[j].y, qq.y, o);
                    o = fmaf(S[j].z, qq.z, o);
                    o = fmaf(S[j].w, qq.w, o);
                }
#pragma unroll
                for (int m = 1; m < TPR; m <<= 1) o += __shfl_xor_sync(0xffffffffu, o, m);
                if (sub == 0) so[tt][row] = a.q_scale * o;
            }
        }
        if (want_out) {
            __syncthreads();
            for (int e = tid; e < nt * D; e += NT) {
                const int tt = e / D, c = e % D;
                const size_t tok = (size_t)l * a.T + t0 + tt;
                oout[(tok * a.Hv + h) * D + c] = from_f32<Tin>(so[tt][c]);
            }
        }
        if (want_w) {
            __syncthreads();
            if (tid == 0) {
                for (int tt = 0; tt < nt; ++tt) {
                    wsum += sqrtf(su2[tt]);
                    su2[tt] = 0.f;
                }
            }
        }
    }
    if (want_w && tid == 0) a.wnorm[lh] = wsum;

    float num = 0.f, den = 0.f;
#pragma unroll
    for (int j = 0; j < NG; ++j) {
        *reinterpret_cast<float4*>(Srow + 4 * (j * TPR + sub)) = S[j];
        const float dx = S[j].x - S0[j].x, dy = S[j].y - S0[j].y, dz = S[j].z - S0[j].z, dw = S[j].w - S0[j].w;
        num += dx * dx + dy * dy + dz * dz + dw * dw;
        den += S0[j].x * S0[j].x + S0[j].y * S0[j].y + S0[j].z * S0[j].z + S0[j].w * S0[j].w;
    }
    if (a.partials == nullptr) return;
    double dn = num, dd = den;
    // fixed-order xor tree over the lanes that exist (NT < 32 only for d = 16)
#pragma unroll
    for (int m = (NT >= 32 ? 16 : NT / 2); m >= 1; m >>= 1) {
        dn += __shfl_xor_sync(kLanes, dn, m);
        dd += __shfl_xor_sync(kLanes, dd, m);
    }
    constexpr int NW = (NT + 31) / 32;
    if (NT < 32) {   // a single partial warp: the xor tree above already covered its lanes
        if (tid == 0) {
            a.partials[(size_t)lh * 2 + 0] = (float)dn;
            a.partials[(size_t)lh * 2 + 1] = (float)dd;
        }
        return;
    }
    if ((tid & 31) == 0) { red[0][tid >> 5] = dn; red[1][tid >> 5] = dd; }
    __syncthreads();
    if (tid == 0) {
        double sn = 0.0, sd = 0.0;
        for (int w = 0; w < NW; ++w) { sn += red[0][w]; sd += red[1][w]; }
        a.partials[(size_t)lh * 2 + 0] = (float)sn;
        a.partials[(size_t)lh * 2 + 1] = (float)sd;
    }
}

template <typename Tin, int D>
cudaError_t launch_t(const GdnArgs& a, cudaStream_t s) {
    gdn_update_simt_kernel<Tin, D><<<a.L * a.Hv, SimtShape<D>::NT, 0, s>>>(a);
    return cudaGetLastError();
}

template <typename Tin>
cudaError_t launch_d(const GdnArgs& a, cudaStream_t s) {
    switch (a.dk) {
        case 16: return launch_t<Tin, 16>(a, s);
        case 32: return launch_t<Tin, 32>(a, s);
        case 64: return launch_t<Tin, 64>(a, s);
        case 128: return launch_t<Tin, 128>(a, s);
        default: return cudaErrorInvalidValue;
    }
}

}  // namespace

cudaError_t launch_gdn_update_simt(const GdnArgs& a, cudaStream_t s) {
    return a.dtype == DELTAS_BF16 ? launch_d<__nv_bfloat16>(a, s) : launch_d<float>(a, s);
}

}  // namespace deltas
