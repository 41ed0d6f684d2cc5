// Gated delta rule over one chunk on the Blackwell tensor cores (tcgen05 + TMEM + TMA), d = 128,
// bfloat16 k/v, fp32 state, with the state-drift partials fused in.
//
// Paper: Sec. 3.2, Eq. 1/2 (the recurrence) and Eq. 3 (drift numerator / denominator per layer
// and head).  The chunk is processed in tiles of C = 64 tokens with the chunkwise (WY) form of
// Eq. 1: with G the inclusive cumulative log-decay inside the tile, gamma = exp(G),
//   A[t][i] = beta_t exp(G_t - G_i) k_t.k_i  (i < t),   T = (I + A)^-1 diag(beta),
//   X = K S0^T,   U = T (V - diag(gamma) X),
//   S_C = gamma_C S0 + U~^T K,   U~[t] = exp(G_C - G_t) U[t].
// Padded tokens of a ragged last tile carry k = v = 0, g = 0, beta = 0 and change nothing.
//
// One persistent CTA per SM takes (layer, value head) pairs in turn, each for the whole chunk;
// the tiles of its heads form one pipeline, so a head's loads and T builds start while the
// previous head drains.  A head's state lives in TMEM from its first tile to its last and
// S_before stays in shared memory, so the state is read from and written to HBM exactly once and
// the drift needs no second pass over it.
//
// Precision.  Keys and values are exact in bfloat16.  The state never leaves fp32 inside the
// tile loop: TMEM holds S~ with S = sig S~, and X = K S0^T reads S~ straight from TMEM as the A
// operand of a kind::tf32 product (B = K converted to fp32 in shared memory); the hardware keeps
// 10 mantissa bits of S~ (a relative error below 2^-10 per element), an error that reaches the
// state only through the delta correction and decays with it (a CPU simulation of the truncation
// gives a state error vs fp64 of ~2e-4 at the slowest decay the inputs use, 5e-6 at a typical
// one).  The other products take a
// two-term bfloat16 split (x = hi + lo, hi = bf16(x), lo = bf16(x - hi)) of their state-side
// operand.  With X~ = -diag(gamma) X:
//   X^T  = S0 K^T                   S~ (tf32, from TMEM) K32^T                    1 MMA group
//   U^T  = V^T T^T + X~^T T^T        V^T (Thi + Tlo) + X~hi (Thi + Tlo) + X~lo Thi  5 MMA groups
//   S   += U~^T K                   (U~hi + U~lo) K                              2 MMA groups
//   K K^T                           exact inputs                                 1 MMA group
// All products accumulate in fp32 in TMEM.
//
// Deferred decay: the tile decay gamma_C is folded into the scalar sig instead of a pass that
// multiplies S by gamma_C; X~ is scaled by sig and U~ by 1 / (gamma_C sig) so that MMA_S adds
// onto S~ directly.  When sig gamma_C would fall below 2^-30 the tile writes gamma_C sig S~ back
// into TMEM and sig restarts at 1, so 1 / sig stays far from the fp32 range limit.  The head's
// last tile multiplies by sig when it reads the state out.
//
// Operand placement: the state-side operands (S~, X~, U~) are A operands read straight from TMEM
// (written there by tcgen05.st), so the only operands streamed from shared memory are K, V and T.
// Shared-memory bandwidth is the resource the tensor pipe and the CUDA-core warps share, and A
// tiles of 128 rows re-read for every N = 64 product would otherwise saturate it.
//
// Warp roles (17 warps):
//   0-7   state chain: per tile, X~ split, U~ split (TMEM <-> registers), next tile's K -> fp32,
//         and at a head's first / last tile the state load / store and the drift partials
//   8-15  T builders: K K^T -> A -> (I + A)^-1 by 16 / 32 / 64 blocks -> T (hi, lo), a tile ahead
//         of the chain (T depends on k, g, beta only)
//   16    TMEM allocation, TMA loads and every tcgen05.mma (the warp stays converged; elect.sync
//         picks the issuing lane)
// Roles hand work to each other through mbarriers only.  Every wait is bounded; a wait that runs
// out records DELTAS_ERR_TIMEOUT, raises a CTA-wide abort flag so the other roles stop waiting,
// and the CTA drains its MMAs and loads before freeing TMEM.
// TMEM (512 columns, M = 128 lanes = d_v): S~ [0,128) (fp32), X [256,320) (fp32, then X~ hi / lo
// packed in place), U [320,384) (likewise U~), K K^T of even / odd tiles [384,448) / [448,512);
// [128,256) is unused.
#include <algorithm>

#include "internal.cuh"
#include "tc_ptx.cuh"

namespace deltas {
namespace {

using namespace tc;

constexpr int kC = 64;                 // tokens per tile
constexpr int kD = 128;                // head dim (d_k = d_v)
constexpr int kChain = 256;            // warps 0-7
constexpr int kTB = 256;               // warps 8-15
constexpr int kThreads = kChain + kTB + 32;
constexpr int kCtlWarp = 16;
constexpr uint32_t kTmemCols = 512;
constexpr uint32_t TM_S = 0, TM_X = 256, TM_U = 320, TM_KK = 384;  // K K^T: 2 x 64; [128,256) unused

constexpr int FA_S = 68;               // fp32 row stride of A: 16-byte rows; a 16-byte access by 8 threads
                                       // of 8 consecutive rows hits 8 distinct bank groups
constexpr int FX_S = 68;               // fp32 row stride of X^-1 (16-byte aligned rows for float4 reads)

// shared-memory map (bytes from a 1024-aligned base)
constexpr uint32_t SM_K = 0;                      // 3 x 16 KB: K tile, 2 column blocks (d 0-63, 64-127) x 64 rows x 128 B
constexpr uint32_t SM_V = 49152;                  // 16 KB: V tile, same layout
constexpr uint32_t SM_T = 65536;                  // hi 8 KB, lo 8 KB: T, 64 rows (t) x 64 (i)
constexpr uint32_t SM_K32 = 81920;                // 32 KB: K tile in fp32 (the tf32 B operand of X), 4 column
                                                  // blocks (32 dims) x 64 rows x 128 B, SW128
constexpr uint32_t SM_SB = 114688;                // 64 KB: S_before fp32, 4 column blocks x 128 rows x 128 B, SW128
constexpr uint32_t SM_FA = 180224;                // fp32 [64][FA_S]
constexpr uint32_t SM_FX = SM_FA + 64 * FA_S * 4; // fp32 [64][FX_S]
constexpr uint32_t SM_TMP = SM_FX + 64 * FX_S * 4;// fp32 [32][33]
constexpr uint32_t SM_CG = SM_TMP + 32 * 33 * 4;  // chain tile constants, 3 buffers x (-gamma[64], del[64], gamma_C)
constexpr uint32_t SM_TG = SM_CG + 3 * 132 * 4;   // T-builder constants, 2 buffers (tile parity) x
                                                  // (G2[64], beta[64], row[64], col[64], flag)
constexpr uint32_t kTgFloats = 260;
constexpr uint32_t SM_BYTES = SM_TG + 2 * kTgFloats * 4;
constexpr uint32_t kSmemAlloc = SM_BYTES + 1024;
static_assert(SM_TG % 16 == 0, "beta must be 16-byte aligned");
static_assert(kSmemAlloc <= 232448, "shared memory budget");

constexpr float kLog2e = 1.4426950408889634f;
constexpr float kSigMin = 9.313225746154785e-10f;   // 2^-30: smallest deferred decay of the state

// S_before: the head's [d_v][d_k] fp32 state as four column blocks of 32 floats, each 128 rows x
// 128 bytes with the 128-byte swizzle (16-byte chunk ^ (row & 7)) that TMA writes and reads; eight
// threads reading chunk c of eight consecutive rows (one row per thread) hit distinct banks.
// Float offset of 16-byte chunk `chunk` (0..31) of row `row`:
__device__ __forceinline__ int sb_idx(int row, int chunk) {
    return (chunk >> 3) * 4096 + row * 32 + (((chunk & 7) ^ (row & 7)) << 2);
}

struct TcArgs {
    int L, Hk, Hv, T, n_tiles;
    float* state;
    float* partials;
    const float* g;
    const float* beta;
    int32_t* status;
};

// Where a global tile lies: tile jt of head lh = (layer l, value head h), key head kh.  Each role
// walks the tiles in order; a step costs integer divisions only when it crosses into the next head.
struct TileCursor {
    int jt, lh, l, h, kh;
    __device__ __forceinline__ void set_head(int head, const TcArgs& a) {
        lh = head; l = head / a.Hv; h = head - l * a.Hv;
        kh = (int)(((long long)h * a.Hk) / a.Hv);
    }
    __device__ __forceinline__ void init(const TcArgs& a) { jt = 0; set_head((int)blockIdx.x, a); }
    __device__ __forceinline__ void next(int n, const TcArgs& a) {
        if (++jt == n) { jt = 0; set_head(lh + (int)gridDim.x, a); }
    }
};

__device__ __forceinline__ void named_sync(int id, int n) {
    asm volatile("bar.sync %0, %1;" :: "r"(id), "r"(n) : "memory");
}

// Barrier over `n` threads that also returns the OR of `flag` over them (uniform result).
__device__ __forceinline__ bool named_sync_or(int id, int n, bool flag) {
    uint32_t out;
    asm volatile("{\n\t.reg .pred p, q;\n\t"
                 "setp.ne.u32 q, %3, 0;\n\t"
                 "bar.red.or.pred p, %1, %2, q;\n\t"
                 "selp.u32 %0, 1, 0, p;\n\t}"
                 : "=r"(out) : "r"(id), "r"(n), "r"((uint32_t)flag) : "memory");
    return out != 0;
}

__device__ __forceinline__ uint32_t pack_bf16x2(float a, float b) {
    __nv_bfloat162 v = __floats2bfloat162_rn(a, b);
    return *reinterpret_cast<uint32_t*>(&v);
}

// x[0..7] -> hi = bf16(x), lo = bf16(x - hi), 8 packed values each
__device__ __forceinline__ void split8(const float* x, uint4& hi, uint4& lo) {
    uint32_t h[4], l[4];
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        const __nv_bfloat162 hh = __floats2bfloat162_rn(x[2 * i], x[2 * i + 1]);
        const float2 hf = __bfloat1622float2(hh);
        h[i] = *reinterpret_cast<const uint32_t*>(&hh);
        l[i] = pack_bf16x2(x[2 * i] - hf.x, x[2 * i + 1] - hf.y);
    }
    hi = make_uint4(h[0], h[1], h[2], h[3]);
    lo = make_uint4(l[0], l[1], l[2], l[3]);
}

// (a, b) -> packed bf16 hi = (bf16(a), bf16(b)) and lo = (bf16(a - hi_a), bf16(b - hi_b)),
// a in the low half (the TMEM A-operand packing: even k low)
__device__ __forceinline__ void split2(float a, float b, uint32_t& hi, uint32_t& lo) {
    const __nv_bfloat162 hh = __floats2bfloat162_rn(a, b);
    const float2 hf = __bfloat1622float2(hh);
    hi = *reinterpret_cast<const uint32_t*>(&hh);
    lo = pack_bf16x2(a - hf.x, b - hf.y);
}

// 2^x with the hardware approximation (relative error about 2^-22)
__device__ __forceinline__ float fast_exp2(float x) {
    float y;
    asm("ex2.approx.f32 %0, %1;" : "=f"(y) : "f"(x));
    return y;
}

// All lanes of a converged warp wait; the result is the same on every lane (false if any lane's
// wait ran out), so the warp stays converged for the elect.sync that follows.
__device__ __forceinline__ bool warp_wait(uint64_t* bar, uint32_t parity, uint64_t budget_ns,
                                          const volatile int* abort) {
    const bool ok = mbar_wait_or_abort(bar, parity, budget_ns, abort);
    return __all_sync(0xffffffffu, ok) != 0;
}

__device__ __forceinline__ void fail(int32_t* status, volatile int* abort, int where) {
    record_status(status, DELTAS_ERR_TIMEOUT, where);
    *abort = 1;
}

__global__ void __launch_bounds__(kThreads, 1)
gdn_update_tc_kernel(const __grid_constant__ CUtensorMap kmap, const __grid_constant__ CUtensorMap vmap,
                     const __grid_constant__ CUtensorMap smap, TcArgs a)
{
    extern __shared__ uint8_t smem_raw[];
    uint8_t* sm = smem_raw + ((1024 - (smem_u32(smem_raw) & 1023)) & 1023);
    // TMA -> MMA: K buffers, V buffer.  MMA -> roles: kk, x, u, s.  roles -> MMA: ready flags.
    __shared__ uint64_t mb_tk[3], mb_tv, mb_kk[2], mb_x, mb_u, mb_s, mb_sready, mb_xready, mb_uready, mb_tready, mb_fin;
    __shared__ uint64_t mb_cready[3];                  // chain tile constants of tile t in buffer t % 3
    __shared__ uint64_t mb_st;                         // a head's state landed in S_before
    __shared__ uint32_t s_tmem;
    __shared__ int s_abort;
    __shared__ double s_red[2][8];
    volatile int* abort_flag = &s_abort;

    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int n = a.n_tiles;
    // Persistent CTA: it owns heads blockIdx.x, blockIdx.x + gridDim.x, ...  Their tiles form one
    // sequence J = head slot * n + tile, over which every role keeps its barrier phases, so the
    // next head's loads and T builds overlap the current head's last tiles.
    const int n_heads = a.L * a.Hv;
    const int NJ = ((n_heads - (int)blockIdx.x + (int)gridDim.x - 1) / (int)gridDim.x) * n;

    if (warp == kCtlWarp) {
        tmem_alloc(&s_tmem, kTmemCols);
        tmem_relinquish();
        if (lane == 0) {
            mbar_init(&mb_tk[0], 1); mbar_init(&mb_tk[1], 1); mbar_init(&mb_tk[2], 1); mbar_init(&mb_tv, 1);
            mbar_init(&mb_kk[0], 1); mbar_init(&mb_kk[1], 1);
            mbar_init(&mb_x, 1); mbar_init(&mb_u, 1); mbar_init(&mb_s, 1);
            mbar_init(&mb_sready, kChain); mbar_init(&mb_xready, kChain); mbar_init(&mb_uready, kChain);
            mbar_init(&mb_tready, kTB); mbar_init(&mb_fin, 1);
            mbar_init(&mb_cready[0], 1); mbar_init(&mb_cready[1], 1); mbar_init(&mb_cready[2], 1);
            mbar_init(&mb_st, 1);
            fence_barrier_init();
            prefetch_tensormap(&kmap);
            prefetch_tensormap(&vmap);
            prefetch_tensormap(&smap);
        }
    }
    if (tid == 0) s_abort = 0;
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tm = s_tmem;

    if (warp == kCtlWarp) {
        // =========================================================== TMA + MMA issue (whole warp,
        // converged; elect.sync picks the issuing lane)
        {
            TileCursor kc, vc;                         // next K / V tile to load (loaded in order)
            kc.init(a); vc.init(a);
            auto load_k = [&](int J) {                 // K tile of global tile J -> buffer J % 3
                const int b = J % 3;
                if (elect_one()) {
                    uint8_t* dst = sm + SM_K + b * 16384;
                    mbar_arrive_expect_tx(&mb_tk[b], 16384);
                    tma_load_4d(dst, &kmap, &mb_tk[b], 0, kc.kh, kc.jt * kC, kc.l);
                    tma_load_4d(dst + 8192, &kmap, &mb_tk[b], 64, kc.kh, kc.jt * kC, kc.l);
                }
                __syncwarp();
                kc.next(n, a);
            };
            auto load_v = [&]() {
                if (elect_one()) {
                    mbar_arrive_expect_tx(&mb_tv, 16384);
                    tma_load_4d(sm + SM_V, &vmap, &mb_tv, 0, vc.h, vc.jt * kC, vc.l);
                    tma_load_4d(sm + SM_V + 8192, &vmap, &mb_tv, 64, vc.h, vc.jt * kC, vc.l);
                }
                __syncwarp();
                vc.next(n, a);
            };
            auto mma_kk = [&](int tile) {
                // K K^T into the K K^T buffer of the tile's parity.  M = 128: rows 64..127 of A read
                // the next 8 KB of shared memory (valid, ignored output).
                const uint8_t* sK = sm + SM_K + (tile % 3) * 16384;
                const uint32_t id = idesc_bf16(128, 64, 0, 0);
#pragma unroll
                for (int s = 0; s < 8; ++s) {
                    const uint64_t d = sdesc_sw128(smem_u32(sK + (s >> 2) * 8192 + (s & 3) * 32), 16, 1024);
                    mma_bf16(tm + TM_KK + 64 * (tile & 1), d, d, id, s > 0);
                }
                mma_commit(&mb_kk[tile & 1]);
            };
            int kp[3] = {-1, -1, -1};                  // tile whose K load is in flight, per buffer
            int v_pending = 0;
            load_k(0); kp[0] = 0;
            if (NJ > 1) { load_k(1); kp[1] = 1; }
            load_v();
            bool ok = warp_wait(&mb_tk[0], 0, kWaitBudgetNs, abort_flag);
            if (!ok) fail(a.status, abort_flag, 1);
            if (ok) { kp[0] = -1; mma_kk(0); }
            for (int j = 0; ok && j < NJ; ++j) {          // j: global tile index
                const uint8_t* sK = sm + SM_K + (j % 3) * 16384;
                // tile j ready for X: the fp32 copy of K(j) is written and, at a head's first tile, the
                // state is in TMEM (otherwise MMA_S(j-1), issued before, produces it in pipe order)
                if (!warp_wait(&mb_sready, j & 1, kWaitBudgetNs, abort_flag)) { fail(a.status, abort_flag, 2); break; }
                tc_fence_after();
                {   // X~^T = S~ K^T: A = the fp32 state straight from TMEM read as tf32 (8 columns per
                    // K = 8 step), B = K in fp32
                    const uint32_t id = idesc_tf32(128, 64);
                    const uint8_t* k32 = sm + SM_K32;
#pragma unroll
                    for (int s = 0; s < 16; ++s) {
                        const uint64_t bd = sdesc_sw128(smem_u32(k32 + (s >> 2) * 8192 + (s & 3) * 32), 16, 1024);
                        mma_tf32_ta(tm + TM_X, tm + TM_S + 8 * s, bd, id, s != 0);
                    }
                    mma_commit(&mb_x);
                }
                if (j + 1 < NJ) {                      // K K^T of the next tile, for the T builders
                    if (!warp_wait(&mb_tk[(j + 1) % 3], ((j + 1) / 3) & 1, kWaitBudgetNs, abort_flag)) {
                        fail(a.status, abort_flag, 4); break;
                    }
                    kp[(j + 1) % 3] = -1;
                    mma_kk(j + 1);
                }
                if (!warp_wait(&mb_tready, j & 1, kWaitBudgetNs, abort_flag)) { fail(a.status, abort_flag, 3); break; }
                if (!warp_wait(&mb_xready, j & 1, kWaitBudgetNs, abort_flag)) { fail(a.status, abort_flag, 5); break; }
                if (!warp_wait(&mb_tv, j & 1, kWaitBudgetNs, abort_flag)) { fail(a.status, abort_flag, 6); break; }
                v_pending = -1;
                tc_fence_after();
                {   // U^T = V^T T^T + X~^T T^T   (X~ = -diag(gamma) X, hi / lo packed in place in X)
                    const uint8_t* tb = sm + SM_T;
                    const uint32_t id_v = idesc_bf16(128, 64, 1, 0);      // A = V tile read MN-major
                    const uint32_t id_x = idesc_bf16(128, 64, 0, 0);      // A = X~ from TMEM
#pragma unroll
                    for (int part = 0; part < 5; ++part) {
                        const uint8_t* sb = tb + ((part == 1 || part == 3) ? 8192 : 0);
#pragma unroll
                        for (int s = 0; s < 4; ++s) {
                            const uint64_t bd = sdesc_sw128(smem_u32(sb + s * 32), 16, 1024);
                            const uint32_t acc = (part | s) != 0;
                            if (part < 2) {
                                mma_bf16(tm + TM_U, sdesc_sw128(smem_u32(sm + SM_V + s * 2048), 8192, 1024), bd, id_v, acc);
                            } else {
                                // tokens 16s..16s+15: column block s/2 of the X region, hi then lo
                                const uint32_t a = tm + TM_X + 32 * (s >> 1) + 8 * (s & 1) + (part == 4 ? 16 : 0);
                                mma_bf16_ta(tm + TM_U, a, bd, id_x, acc);
                            }
                        }
                    }
                    mma_commit(&mb_u);
                }
                // TMA loads are issued behind MMA groups, never between a wait and the MMAs it
                // releases (a TMA write burst into shared memory slows the issue of a group).
                // K(j+2) reuses the buffer of K(j-1), whose last reader MMA_S(j-1) has completed.
                if (j + 2 < NJ) { load_k(j + 2); kp[(j + 2) % 3] = j + 2; }
                if (!warp_wait(&mb_uready, j & 1, kWaitBudgetNs, abort_flag)) { fail(a.status, abort_flag, 7); break; }
                tc_fence_after();
                {   // S += U~^T K  (A: U~ hi / lo packed in place in U; K read MN-major: N = d_k)
                    const uint32_t id = idesc_bf16(128, 128, 0, 1);
#pragma unroll
                    for (int part = 0; part < 2; ++part) {
#pragma unroll
                        for (int s = 0; s < 4; ++s) {
                            const uint32_t a = tm + TM_U + 32 * (s >> 1) + 8 * (s & 1) + (part == 1 ? 16 : 0);
                            const uint64_t bd = sdesc_sw128(smem_u32(sK + s * 2048), 8192, 1024);
                            mma_bf16_ta(tm + TM_S, a, bd, id, 1);
                        }
                    }
                    mma_commit(&mb_s);
                }
                // V(j+1) into the single V buffer: MMA_U(j), its reader, completed before uready
                if (j + 1 < NJ) { load_v(); v_pending = j + 1; }
            }
            if (__any_sync(0xffffffffu, *abort_flag != 0)) {
                // drain: every MMA this warp issued, and every load still in flight
                mma_commit(&mb_fin);
                mbar_wait(&mb_fin, 0, kWaitBudgetNs);
                for (int b = 0; b < 3; ++b)
                    if (kp[b] >= 0) mbar_wait(&mb_tk[b], (kp[b] / 3) & 1, kWaitBudgetNs);
                if (v_pending >= 0) mbar_wait(&mb_tv, v_pending & 1, kWaitBudgetNs);
            }
        }
        __syncwarp();
    } else if (warp >= 8) {
        // =========================================================== T builders (warps 8-15)
        const int tw = warp - 8, tt = tid - kChain;        // tw in [0, 8), tt in [0, 256)
        float* fA = reinterpret_cast<float*>(sm + SM_FA);
        float* fX = reinterpret_cast<float*>(sm + SM_FX);
        float* fT = reinterpret_cast<float*>(sm + SM_TMP);
        float* cg = reinterpret_cast<float*>(sm + SM_CG);
        float pg[2] = {0.f, 0.f}, pb[2] = {0.f, 0.f};     // g, beta of the next tile (warp 15)
        TileCursor gc;                                     // next tile whose g, beta to load
        gc.init(a);
        auto load_gb = [&]() {                             // g, beta of the next tile (warp 15)
#pragma unroll
            for (int e = 0; e < 2; ++e) {
                const int t = gc.jt * kC + 2 * lane + e;
                const size_t gi = ((size_t)gc.l * a.T + t) * a.Hv + gc.h;
                pg[e] = t < a.T ? a.g[gi] : 0.f;
                pb[e] = t < a.T ? a.beta[gi] : 0.f;
            }
            gc.next(n, a);
        };
        // Decay constants of tile jj from the loaded g, beta (warp 15, one tile ahead of the
        // T build that uses them): the chain's -gamma, exp(G_C - G), gamma_C, and the T builders'
        // G2, beta, row and column factors (buffer jj & 1).
        auto tile_constants = [&](int jj) {
            float* tg = reinterpret_cast<float*>(sm + SM_TG) + (jj & 1) * kTgFloats;
            float gv[2], bv[2];
#pragma unroll
            for (int e = 0; e < 2; ++e) { gv[e] = pg[e]; bv[e] = pb[e]; }
            float incl = gv[0] + gv[1];
#pragma unroll
            for (int m = 1; m < 32; m <<= 1) {
                const float y = __shfl_up_sync(0xffffffffu, incl, m);
                if (lane >= m) incl += y;
            }
            const float G0 = incl - gv[1], G1 = incl;
            const float GC = __shfl_sync(0xffffffffu, incl, 31);
            // the chain's constants of tile jj (3 buffers: the chain is at most two tiles behind
            // the T builders' current tile)
            float* cgam = cg + (jj % 3) * 132;
            cgam[2 * lane] = -expf(G0); cgam[2 * lane + 1] = -expf(G1);
            cgam[64 + 2 * lane] = expf(GC - G0); cgam[64 + 2 * lane + 1] = expf(GC - G1);
            if (lane == 0) cgam[128] = expf(GC);
            const float g20 = G0 * kLog2e, g21 = G1 * kLog2e;
            float lo2 = fminf(g20, g21), hi2 = fmaxf(g20, g21);
#pragma unroll
            for (int m = 16; m >= 1; m >>= 1) {
                lo2 = fminf(lo2, __shfl_xor_sync(0xffffffffu, lo2, m));
                hi2 = fmaxf(hi2, __shfl_xor_sync(0xffffffffu, hi2, m));
            }
            // exp(G_t - G_i) = row_t * col_i with the reference in the middle of the tile's range
            // of G; both factors stay within 2^+-126 when that range spans at most 250 powers of
            // two, otherwise the exponent is taken per entry.
            const float ref = 0.5f * (lo2 + hi2);
            tg[2 * lane] = g20; tg[2 * lane + 1] = g21;
            tg[64 + 2 * lane] = bv[0]; tg[64 + 2 * lane + 1] = bv[1];
            tg[128 + 2 * lane] = bv[0] * fast_exp2(g20 - ref); tg[128 + 2 * lane + 1] = bv[1] * fast_exp2(g21 - ref);
            tg[192 + 2 * lane] = fast_exp2(ref - g20); tg[192 + 2 * lane + 1] = fast_exp2(ref - g21);
            if (lane == 0) reinterpret_cast<int*>(tg)[256] = (hi2 - lo2) <= 250.f;
            fence_async_smem();
            __syncwarp();
            if (lane == 0) mbar_arrive(&mb_cready[jj % 3]);
        };
        // The strictly upper 16 x 16 blocks of X are never written; zeros there let every level
        // run fixed-length (unrolled) loops over the triangular factors.
        for (int e = tt; e < 64 * FX_S; e += kTB) fX[e] = 0.f;
        if (tw == 7 && NJ > 0) {
            load_gb();
            tile_constants(0);
            if (NJ > 1) load_gb();
        }
        for (int j = 0; j < NJ; ++j) {                     // j: global tile index
            if (named_sync_or(3, kTB, *abort_flag)) break;
            const float* tg = reinterpret_cast<const float*>(sm + SM_TG) + (j & 1) * kTgFloats;
            const float* sG2 = tg;                         // G * log2(e)
            const float* sBeta = tg + 64;
            const float* sRow = tg + 128;                  // beta_t 2^(G2_t - ref)
            const float* sCol = tg + 192;                  // 2^(ref - G2_i)
            const int factored = reinterpret_cast<const int*>(tg)[256];
            if (!mbar_wait_or_abort(&mb_kk[j & 1], (j >> 1) & 1, kWaitBudgetNs, abort_flag)) fail(a.status, abort_flag, 8);
            tc_fence_after();
            const int q = warp & 3;
            if (q < 2) {
                // TMEM lanes 0..63 hold K K^T: warps 8/12 rows 0..31, 9/13 rows 32..63; column half
                // (tw >> 2).  All shared-memory reads are made before the first store (the tile
                // constants and A share one buffer).
                const int t = 32 * q + lane, c0 = 32 * (tw >> 2);
                const uint32_t lane_off = (uint32_t)(32 * q) << 16;
                float kk[32], cf[32];
                tmem_ld32(tm + lane_off + TM_KK + 64 * (j & 1) + c0, kk);
                if (factored) {
                    const float rt = sRow[t];
#pragma unroll
                    for (int e = 0; e < 8; ++e) {
                        const float4 v4 = *reinterpret_cast<const float4*>(sCol + c0 + 4 * e);
                        cf[4 * e] = v4.x; cf[4 * e + 1] = v4.y; cf[4 * e + 2] = v4.z; cf[4 * e + 3] = v4.w;
                    }
                    tmem_ld_wait();
#pragma unroll
                    for (int e = 0; e < 32; ++e) kk[e] = (c0 + e < t) ? rt * cf[e] * kk[e] : 0.f;
                } else {
                    const float G2t = sG2[t], bt = sBeta[t];
#pragma unroll
                    for (int e = 0; e < 8; ++e) {
                        const float4 v4 = *reinterpret_cast<const float4*>(sG2 + c0 + 4 * e);
                        cf[4 * e] = v4.x; cf[4 * e + 1] = v4.y; cf[4 * e + 2] = v4.z; cf[4 * e + 3] = v4.w;
                    }
                    tmem_ld_wait();
#pragma unroll
                    for (int e = 0; e < 32; ++e) kk[e] = (c0 + e < t) ? bt * fast_exp2(G2t - cf[e]) * kk[e] : 0.f;
                }
#pragma unroll
                for (int e = 0; e < 8; ++e)
                    *reinterpret_cast<float4*>(fA + t * FA_S + c0 + 4 * e) =
                        make_float4(kk[4 * e], kk[4 * e + 1], kk[4 * e + 2], kk[4 * e + 3]);
            } else if (tw == 7 && j + 1 < NJ) {
                tile_constants(j + 1);                     // the next tile's, off this tile's path
                if (j + 2 < NJ) load_gb();
            }
            tc_fence_before();
            named_sync(3, kTB);
            // level 0: four 16 x 16 diagonal blocks of (I + A)^-1, one column per thread
            if (tt < 64) {
                const int B = tt >> 4, jc = tt & 15, o = 16 * B;
                float x[16];
#pragma unroll
                for (int rr = 0; rr < 16; ++rr) x[rr] = (rr == jc) ? 1.f : 0.f;
#pragma unroll
                for (int rr = 1; rr < 16; ++rr) {
                    float s0 = 0.f, s1 = 0.f;              // two chains: half the dependent FMAs
#pragma unroll
                    for (int c = 0; c < rr; c += 4) {
                        const float4 av = *reinterpret_cast<const float4*>(fA + (o + rr) * FA_S + o + c);
                        s0 = fmaf(av.x, x[c], s0);
                        if (c + 1 < rr) s1 = fmaf(av.y, x[c + 1], s1);
                        if (c + 2 < rr) s0 = fmaf(av.z, x[c + 2], s0);
                        if (c + 3 < rr) s1 = fmaf(av.w, x[c + 3], s1);
                    }
                    if (rr > jc) x[rr] = -(s0 + s1);
                }
#pragma unroll
                for (int rr = 0; rr < 16; ++rr) fX[(o + rr) * FX_S + o + jc] = x[rr];
            }
            named_sync(3, kTB);
            // level 1: X[2p+1][2p] = -X[2p+1][2p+1] (A[2p+1][2p] X[2p][2p]), p = tw >> 2.
            // Fixed-length loops: the zeros of the triangular factors are stored.
            {
                const int p = tw >> 2, cg = 4 * (tw & 3);
                const int ro = 16 * (2 * p + 1), co = 16 * (2 * p);
                const int lo16 = lane & 15, sub = 2 * (lane >> 4);
                float acc0 = 0.f, acc1 = 0.f;             // tmp1[p][lo16][cg + sub + {0,1}]
#pragma unroll
                for (int k4 = 0; k4 < 16; k4 += 4) {
                    const float4 a4 = *reinterpret_cast<const float4*>(fA + (ro + lo16) * FA_S + co + k4);
                    const float av[4] = {a4.x, a4.y, a4.z, a4.w};
#pragma unroll
                    for (int kk4 = 0; kk4 < 4; ++kk4) {
                        const float2 xv = *reinterpret_cast<const float2*>(fX + (co + k4 + kk4) * FX_S + co + cg + sub);
                        acc0 = fmaf(av[kk4], xv.x, acc0);
                        acc1 = fmaf(av[kk4], xv.y, acc1);
                    }
                }
                fT[p * 272 + lo16 * 17 + cg + sub] = acc0;
                fT[p * 272 + lo16 * 17 + cg + sub + 1] = acc1;
                named_sync(3, kTB);
                float o0 = 0.f, o1 = 0.f;                  // rows cg + sub + {0,1}, column lo16
#pragma unroll
                for (int k = 0; k < 16; ++k) {
                    const float tv = fT[p * 272 + k * 17 + lo16];
                    o0 = fmaf(fX[(ro + cg + sub) * FX_S + ro + k], tv, o0);
                    o1 = fmaf(fX[(ro + cg + sub + 1) * FX_S + ro + k], tv, o1);
                }
                fX[(ro + cg + sub) * FX_S + co + lo16] = -o0;
                fX[(ro + cg + sub + 1) * FX_S + co + lo16] = -o1;
            }
            named_sync(3, kTB);
            // level 2: X[32:64][0:32] = -X[32:64][32:64] (A[32:64][0:32] X[0:32][0:32])
            {
                const int g4 = 4 * tw;
                float acc[4] = {0.f, 0.f, 0.f, 0.f};       // tmp2[lane][g4..g4+3]
#pragma unroll
                for (int k4 = 0; k4 < 32; k4 += 4) {
                    const float4 a4 = *reinterpret_cast<const float4*>(fA + (32 + lane) * FA_S + k4);
                    const float av[4] = {a4.x, a4.y, a4.z, a4.w};
#pragma unroll
                    for (int kk4 = 0; kk4 < 4; ++kk4) {
                        const float4 xv = *reinterpret_cast<const float4*>(fX + (k4 + kk4) * FX_S + g4);
                        acc[0] = fmaf(av[kk4], xv.x, acc[0]); acc[1] = fmaf(av[kk4], xv.y, acc[1]);
                        acc[2] = fmaf(av[kk4], xv.z, acc[2]); acc[3] = fmaf(av[kk4], xv.w, acc[3]);
                    }
                }
#pragma unroll
                for (int i = 0; i < 4; ++i) fT[lane * 33 + g4 + i] = acc[i];
                named_sync(3, kTB);
                float o4[4] = {0.f, 0.f, 0.f, 0.f};        // rows 32+g4..32+g4+3, column lane
#pragma unroll
                for (int k = 0; k < 32; k += 4) {
                    const float t0v = fT[(k + 0) * 33 + lane], t1v = fT[(k + 1) * 33 + lane];
                    const float t2v = fT[(k + 2) * 33 + lane], t3v = fT[(k + 3) * 33 + lane];
#pragma unroll
                    for (int i = 0; i < 4; ++i) {
                        const float4 xr = *reinterpret_cast<const float4*>(fX + (32 + g4 + i) * FX_S + 32 + k);
                        o4[i] = fmaf(xr.x, t0v, o4[i]); o4[i] = fmaf(xr.y, t1v, o4[i]);
                        o4[i] = fmaf(xr.z, t2v, o4[i]); o4[i] = fmaf(xr.w, t3v, o4[i]);
                    }
                }
#pragma unroll
                for (int i = 0; i < 4; ++i) fX[(32 + g4 + i) * FX_S + lane] = -o4[i];
            }
            // the single T buffer is free once MMA_U(j-1) has read it (it completes long before this
            // point in steady state; MMA_U(j) cannot complete before T(j) is written, so the
            // barrier is never two phases ahead)
            if (j > 0 && !mbar_wait_or_abort(&mb_u, (j - 1) & 1, kWaitBudgetNs, abort_flag)) fail(a.status, abort_flag, 15);
            named_sync(3, kTB);
            // T = X diag(beta) (upper part zero), split into the B operand buffer
            {
                uint8_t* tb = sm + SM_T;
                uint4 vh[2], vl[2];
                int tr[2], cr[2];
#pragma unroll
                for (int m = 0; m < 2; ++m) {
                    const int e = tt + kTB * m;
                    const int t = e >> 3, c8 = e & 7;
                    const float4 x0 = *reinterpret_cast<const float4*>(fX + t * FX_S + 8 * c8);
                    const float4 x1 = *reinterpret_cast<const float4*>(fX + t * FX_S + 8 * c8 + 4);
                    const float4 b0 = *reinterpret_cast<const float4*>(sBeta + 8 * c8);
                    const float4 b1 = *reinterpret_cast<const float4*>(sBeta + 8 * c8 + 4);
                    const float xs[8] = {x0.x * b0.x, x0.y * b0.y, x0.z * b0.z, x0.w * b0.w,
                                         x1.x * b1.x, x1.y * b1.y, x1.z * b1.z, x1.w * b1.w};
                    float x[8];
#pragma unroll
                    for (int k = 0; k < 8; ++k) x[k] = (8 * c8 + k <= t) ? xs[k] : 0.f;
                    split8(x, vh[m], vl[m]);
                    tr[m] = t; cr[m] = c8;
                }
#pragma unroll
                for (int m = 0; m < 2; ++m) {
                    *reinterpret_cast<uint4*>(tb + sw128_offset(tr[m], cr[m])) = vh[m];
                    *reinterpret_cast<uint4*>(tb + 8192 + sw128_offset(tr[m], cr[m])) = vl[m];
                }
            }
            fence_async_smem();
            mbar_arrive(&mb_tready);
        }
    } else {
        // =========================================================== state chain (warps 0-7)
        const int q = warp & 3, wg = warp >> 2;
        const int r = 32 * q + lane;                       // row of S (value index)
        const uint32_t lane_off = (uint32_t)(32 * q) << 16;
        const uint32_t cS = TM_S + 64 * wg;                // this thread's 64 state columns
        float* sbefore = reinterpret_cast<float*>(sm + SM_SB);   // swizzled rows, see sb_idx
        float* cg = reinterpret_cast<float*>(sm + SM_CG);
        // a head's state (128 rows of the state viewed as [L * Hv * d_v][d_k]) into S_before by TMA,
        // issued by thread 0 of the chain, completing on mb_st
        int st_issued = 0, st_seen = 0;                    // state loads issued / waited for (uniform)
        auto load_state = [&](int lh) {
            ++st_issued;
            if (tid == 0) {
                mbar_arrive_expect_tx(&mb_st, kD * kD * 4);
#pragma unroll
                for (int b = 0; b < 4; ++b) tma_load_2d(sbefore + 4096 * b, &smap, &mb_st, 32 * b, lh * kD);
            }
        };
        if (NJ > 0) load_state((int)blockIdx.x);
        TileCursor cc;                                     // the chain's tile
        cc.init(a);
        // K(jj) bf16 (TMA tile, buffer jj % 3) -> fp32 copy for the tf32 X product.  Called between
        // MMA_X(jj-1), the last reader of the copy, and the ready signal of tile jj.
        auto k_to_fp32 = [&](int jj) -> bool {
            const bool ok = mbar_wait_or_abort(&mb_tk[jj % 3], (jj / 3) & 1, kWaitBudgetNs, abort_flag);
            const uint8_t* kb = sm + SM_K + (jj % 3) * 16384;
            uint8_t* k32 = sm + SM_K32;
#pragma unroll
            for (int u = 0; u < 4; ++u) {                  // 64 rows x 16 chunks of 8 bf16
                const int e = tid + kChain * u;
                const int t = e >> 4, cc16 = e & 15, cb = cc16 >> 3, c = cc16 & 7;
                const uint4 w = *reinterpret_cast<const uint4*>(kb + cb * 8192 + sw128_offset(t, c));
                const uint32_t wv[4] = {w.x, w.y, w.z, w.w};
                float f[8];
#pragma unroll
                for (int i = 0; i < 4; ++i) {
                    f[2 * i] = __uint_as_float(wv[i] << 16);
                    f[2 * i + 1] = __uint_as_float(wv[i] & 0xFFFF0000u);
                }
                // dims 64 cb + 8 c .. + 7: fp32 block 2 cb + c / 4, chunks 2 (c % 4) and 2 (c % 4) + 1
                uint8_t* rowp = k32 + (2 * cb + (c >> 2)) * 8192;
                const int q0 = 2 * (c & 3);
                *reinterpret_cast<float4*>(rowp + sw128_offset(t, q0)) = make_float4(f[0], f[1], f[2], f[3]);
                *reinterpret_cast<float4*>(rowp + sw128_offset(t, q0 + 1)) = make_float4(f[4], f[5], f[6], f[7]);
            }
            fence_async_smem();                            // generic writes -> the tensor core's reads
            return ok;
        };
        float den = 0.f;
        // Deferred decay: TMEM holds S~ with the head's state S = sig * S~.  A tile folds its decay
        // gamma_C into sig (X is rescaled by sig in the X~ pass, U~ by 1 / (gamma_C sig) in the U~
        // pass, so MMA_S accumulates onto S~ with no pass over the state); when sig gamma_C would
        // drop below kSigMin the tile instead writes gamma_C S back into TMEM and sig restarts at 1.
        float sig = 1.f;
        for (int j = 0; j < NJ; ++j) {                     // j: global tile index
            const int lh = cc.lh, jt = cc.jt;              // head and tile within the head
            float* gam = cg + (j % 3) * 132;               // -gamma (written by the T builders)
            float* del = gam + 64;                         // exp(G_C - G)
            if (named_sync_or(2, kChain, *abort_flag)) break;
            if (!mbar_wait_or_abort(&mb_cready[j % 3], (j / 3) & 1, kWaitBudgetNs, abort_flag)) fail(a.status, abort_flag, 13);
            const float gC = gam[128];

            if (jt == 0) {
                // ---- a head's first tile: its state (TMA-loaded into S_before at the previous
                // head's end) into TMEM as S~ with sig = 1, and sum S_before^2
                if (!mbar_wait_or_abort(&mb_st, (j / n) & 1, kWaitBudgetNs, abort_flag)) fail(a.status, abort_flag, 14);
                ++st_seen;
                if (j + n < NJ) {                          // the next head's state towards L2
                    const char* nxt = reinterpret_cast<const char*>(a.state + (size_t)(lh + (int)gridDim.x) * kD * kD);
                    asm volatile("prefetch.L2 [%0];" :: "l"(nxt + 256 * tid) : "memory");
                    asm volatile("prefetch.L2 [%0];" :: "l"(nxt + 256 * tid + 128) : "memory");
                }
#pragma unroll
                for (int half = 0; half < 2; ++half) {
                    float sv[32];
#pragma unroll
                    for (int e = 0; e < 8; ++e) {
                        const float4 x = *reinterpret_cast<const float4*>(sbefore + sb_idx(r, 16 * wg + 8 * half + e));
                        sv[4 * e] = x.x; sv[4 * e + 1] = x.y; sv[4 * e + 2] = x.z; sv[4 * e + 3] = x.w;
                    }
#pragma unroll
                    for (int e = 0; e < 32; ++e) den += sv[e] * sv[e];
                    tmem_st32(tm + lane_off + cS + 32 * half, sv);
                }
                sig = 1.f;
                if (j == 0 && !k_to_fp32(0)) fail(a.status, abort_flag, 16);
                tmem_st_wait();
                tc_fence_before();
                mbar_arrive(&mb_sready);
            }
            const bool rescale = sig * gC < kSigMin;       // uniform over the CTA
            const float x_scale = sig;                     // X = sig * (K S~^T)
            const float u_scale = rescale ? 1.f : 1.f / (gC * sig);

            // ---- X~^T = -X^T diag(gamma): (hi, lo) packed in place over this thread's 32 X columns
            if (!mbar_wait_or_abort(&mb_x, j & 1, kWaitBudgetNs, abort_flag)) fail(a.status, abort_flag, 10);
            tc_fence_after();
            {
                float xv[32];
                tmem_ld32(tm + lane_off + TM_X + 32 * wg, xv);
                tmem_ld_wait();
                uint32_t hi[16], lo[16];
#pragma unroll
                for (int c4 = 0; c4 < 8; ++c4) {
                    float4 g4 = *reinterpret_cast<const float4*>(gam + 32 * wg + 4 * c4);
                    g4.x *= x_scale; g4.y *= x_scale; g4.z *= x_scale; g4.w *= x_scale;
                    split2(g4.x * xv[4 * c4], g4.y * xv[4 * c4 + 1], hi[2 * c4], lo[2 * c4]);
                    split2(g4.z * xv[4 * c4 + 2], g4.w * xv[4 * c4 + 3], hi[2 * c4 + 1], lo[2 * c4 + 1]);
                }
                tmem_st16(tm + lane_off + TM_X + 32 * wg, hi);
                tmem_st16(tm + lane_off + TM_X + 32 * wg + 16, lo);
                tmem_st_wait();
            }
            tc_fence_before();
            mbar_arrive(&mb_xready);

            // ---- while MMA_U runs: rescale S~ if the decay would underflow the deferred scale
            // (MMA_X(j) has read S~; MMA_S(j) waits for uready), and the fp32 copy of K(j+1)
            if (rescale) {
                const float f = gC * sig;
#pragma unroll
                for (int half = 0; half < 2; ++half) {
                    float sv[32];
                    tmem_ld32(tm + lane_off + cS + 32 * half, sv);
                    tmem_ld_wait();
#pragma unroll
                    for (int e = 0; e < 32; ++e) sv[e] *= f;
                    tmem_st32(tm + lane_off + cS + 32 * half, sv);
                }
                tmem_st_wait();
            }
            if (j + 1 < NJ && !k_to_fp32(j + 1)) fail(a.status, abort_flag, 16);

            // ---- U~^T = U^T diag(exp(G_C - G)) / (gamma_C sig): (hi, lo) packed in place over U
            if (!mbar_wait_or_abort(&mb_u, j & 1, kWaitBudgetNs, abort_flag)) fail(a.status, abort_flag, 11);
            tc_fence_after();
            {
                float uv[32];
                tmem_ld32(tm + lane_off + TM_U + 32 * wg, uv);
                tmem_ld_wait();
                uint32_t hi[16], lo[16];
#pragma unroll
                for (int c4 = 0; c4 < 8; ++c4) {
                    float4 d4 = *reinterpret_cast<const float4*>(del + 32 * wg + 4 * c4);
                    d4.x *= u_scale; d4.y *= u_scale; d4.z *= u_scale; d4.w *= u_scale;
                    split2(uv[4 * c4] * d4.x, uv[4 * c4 + 1] * d4.y, hi[2 * c4], lo[2 * c4]);
                    split2(uv[4 * c4 + 2] * d4.z, uv[4 * c4 + 3] * d4.w, hi[2 * c4 + 1], lo[2 * c4 + 1]);
                }
                tmem_st16(tm + lane_off + TM_U + 32 * wg, hi);
                tmem_st16(tm + lane_off + TM_U + 32 * wg + 16, lo);
                tmem_st_wait();
            }
            tc_fence_before();
            mbar_arrive(&mb_uready);
            sig = rescale ? 1.f : gC * sig;
            // the next tile of this head may start X as soon as MMA_S(j) is queued
            if (jt < n - 1) mbar_arrive(&mb_sready);

            if (jt == n - 1) {
                // ---- epilogue of the head: S_after -> HBM, drift partials against S_before
                const bool ok = mbar_wait_or_abort(&mb_s, j & 1, kWaitBudgetNs, abort_flag);
                if (!ok) fail(a.status, abort_flag, 12);
                tc_fence_after();
                float num = 0.f;
                if (ok) {
                    // S_after = sig S~ replaces S_before in shared memory (each thread its own row) ...
#pragma unroll
                    for (int half = 0; half < 2; ++half) {
                        float sv[32];
                        tmem_ld32(tm + lane_off + cS + 32 * half, sv);
                        tmem_ld_wait();
#pragma unroll
                        for (int e = 0; e < 32; ++e) sv[e] *= sig;
#pragma unroll
                        for (int e = 0; e < 8; ++e) {
                            float4* p = reinterpret_cast<float4*>(sbefore + sb_idx(r, 16 * wg + 8 * half + e));
                            const float4 b = *p;
                            const float d0 = sv[4 * e] - b.x, d1 = sv[4 * e + 1] - b.y;
                            const float d2 = sv[4 * e + 2] - b.z, d3 = sv[4 * e + 3] - b.w;
                            num += d0 * d0 + d1 * d1 + d2 * d2 + d3 * d3;
                            *p = make_float4(sv[4 * e], sv[4 * e + 1], sv[4 * e + 2], sv[4 * e + 3]);
                        }
                    }
                }
                tc_fence_before();
                fence_async_smem();
                // ... and goes to HBM by TMA; once TMA has read it out, the next head's state
                // comes in
                if (named_sync_or(2, kChain, !ok)) break;
                if (tid == 0) {
#pragma unroll
                    for (int b = 0; b < 4; ++b) tma_store_2d(&smap, sbefore + 4096 * b, 32 * b, lh * kD);
                    bulk_commit();
                    bulk_wait_read0();
                }
                if (j + 1 < NJ) load_state(lh + (int)gridDim.x);
                // partial sums: float within a warp (the FP64 pipe is slow), double across warps
                float fn = num, fd = den;
#pragma unroll
                for (int m = 16; m >= 1; m >>= 1) {
                    fn += __shfl_xor_sync(0xffffffffu, fn, m);
                    fd += __shfl_xor_sync(0xffffffffu, fd, m);
                }
                if (lane == 0) { s_red[0][warp] = fn; s_red[1][warp] = fd; }
                const bool any_fail = named_sync_or(2, kChain, !ok);
                if (tid == 0 && !any_fail && a.partials != nullptr) {
                    double sn = 0.0, sd = 0.0;
                    for (int w = 0; w < 8; ++w) { sn += s_red[0][w]; sd += s_red[1][w]; }
                    a.partials[(size_t)lh * 2 + 0] = (float)sn;
                    a.partials[(size_t)lh * 2 + 1] = (float)sd;
                }
                if (any_fail) break;
                den = 0.f;
            }
            cc.next(n, a);
        }
        if (tid == 0) {
            bulk_wait0();                                  // the last state store is complete
            // abort path: a state load issued but not waited for lands before the CTA ends
            if (st_issued > st_seen) mbar_wait(&mb_st, (st_issued - 1) & 1, kWaitBudgetNs);
        }
    }

    tc_fence_before();
    __syncthreads();
    if (warp == kCtlWarp) {
        tc_fence_after();
        tmem_dealloc(tm, kTmemCols);
    }
}

typedef CUresult (*EncodeTiledFn)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*, const cuuint64_t*,
                                  const cuuint64_t*, const cuuint32_t*, const cuuint32_t*, CUtensorMapInterleave,
                                  CUtensorMapSwizzle, CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

EncodeTiledFn encode_fn() {
    static EncodeTiledFn fn = nullptr;
    static bool tried = false;
    if (!tried) {
        tried = true;
        cudaDriverEntryPointQueryResult q;
        void* p = nullptr;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) == cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            fn = reinterpret_cast<EncodeTiledFn>(p);
    }
    return fn;
}

// [L][T][H][128] bfloat16 as a 4-D map (d, H, T, L): a box of 64 features x 1 head x 64 tokens,
// 128-byte swizzle; tokens past T read as zero.
bool make_map(CUtensorMap* map, const void* base, int L, int T, int H) {
    EncodeTiledFn enc = encode_fn();
    if (!enc) return false;
    cuuint64_t dims[4] = {(cuuint64_t)kD, (cuuint64_t)H, (cuuint64_t)T, (cuuint64_t)L};
    cuuint64_t strides[3] = {(cuuint64_t)kD * 2, (cuuint64_t)H * kD * 2, (cuuint64_t)T * H * kD * 2};
    cuuint32_t box[4] = {64, 1, (cuuint32_t)kC, 1};
    cuuint32_t es[4] = {1, 1, 1, 1};
    return enc(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 4, const_cast<void*>(base), dims, strides, box, es,
               CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
               CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// The state [L * Hv * 128][128] fp32 as a 2-D map: a box of 32 columns x 128 rows (one column block
// of one head), 128-byte swizzle.
bool make_state_map(CUtensorMap* map, void* base, int heads) {
    EncodeTiledFn enc = encode_fn();
    if (!enc) return false;
    cuuint64_t dims[2] = {(cuuint64_t)kD, (cuuint64_t)heads * kD};
    cuuint64_t strides[1] = {(cuuint64_t)kD * 4};
    cuuint32_t box[2] = {32, (cuuint32_t)kD};
    cuuint32_t es[2] = {1, 1};
    return enc(map, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 2, base, dims, strides, box, es,
               CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
               CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

}  // namespace

bool gdn_tc_supported(const GdnArgs& a) {
    return a.dk == kD && a.dv == kD && a.dtype == DELTAS_BF16 && a.out == nullptr && a.T > 0 &&
           (long long)a.L * a.Hv * kD < (1ll << 31) && encode_fn() != nullptr;   // TMA row coordinate
}

cudaError_t launch_gdn_update_tc(const GdnArgs& a, cudaStream_t s) {
    CUtensorMap kmap, vmap, smap;
    if (!make_map(&kmap, a.k, a.L, a.T, a.Hk) || !make_map(&vmap, a.v, a.L, a.T, a.Hv) ||
        !make_state_map(&smap, a.state, a.L * a.Hv))
        return cudaErrorInvalidValue;
    static int configured_device = -1;
    int dev = 0;
    cudaGetDevice(&dev);
    if (configured_device != dev) {
        cudaError_t e = cudaFuncSetAttribute(gdn_update_tc_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                             (int)kSmemAlloc);
        if (e != cudaSuccess) return e;
        configured_device = dev;
    }
    TcArgs t;
    t.L = a.L; t.Hk = a.Hk; t.Hv = a.Hv; t.T = a.T; t.n_tiles = (a.T + kC - 1) / kC;
    t.state = a.state; t.partials = a.partials; t.g = a.g; t.beta = a.beta; t.status = a.status;
    // one persistent CTA per SM (the kernel needs the whole SM: 512 TMEM columns, ~206 KB of
    // shared memory); each takes every grid-th head
    const int grid = std::min(a.L * a.Hv, device_sm_count());
    gdn_update_tc_kernel<<<grid, kThreads, kSmemAlloc, s>>>(kmap, vmap, smap, t);
    return cudaGetLastError();
}

}  // namespace deltas
