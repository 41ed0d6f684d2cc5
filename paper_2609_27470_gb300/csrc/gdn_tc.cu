// Gated delta rule over one chunk on the Blackwell tensor cores (tcgen05 + TMEM + TMA), d = 128,
// bfloat16 k/v, fp32 state, with the state-drift partials fused in: one persistent kernel.
//
// Paper: Sec. 3.2, Eq. 1/2 (the recurrence) and Eq. 3 (drift numerator / denominator per layer
// and head).  The chunk is processed in sub-tiles of C = 32 tokens with the chunkwise (WY) form of
// Eq. 1.  Inside a sub-tile let G be the inclusive cumulative log-decay, gamma_t = exp(G_t),
// gamma_C = exp(G_{C-1}), delta_t = gamma_C / gamma_t <= 1, and X = K S0^T (row t: S0 k_t).  With
//   A[t][i] = beta_t (gamma_t / gamma_i) k_t.k_i  (i < t),   U = (I + A)^-1 diag(beta) (V - diag(gamma) X)
// the state after the sub-tile is S_C = gamma_C S0 + sum_t delta_t u_t k_t^T.  The decay factors
// out of the triangular solve by a diagonal similarity, I + A = diag(gamma) (I + diag(beta) L)
// diag(gamma)^-1 with L the strictly lower part of K K^T, so with the decay-free
//   N_beta = (I + diag(beta) L)^-1 diag(beta)
// the decayed writes are  U~ = diag(delta) U = N_beta (diag(delta) V - gamma_C X):  every decay
// factor the kernel uses is at most 1, and the inverse depends on k and beta only.
//
// Work split inside one CTA (one per SM, persistent over (layer, value head) slots):
//   producer  (4 warps, two groups of two; group g takes the sub-tiles of parity g): K K^T of a
//             64-token tile comes from the tensor core; each group forms diag(beta) L of its
//             sub-tile, inverts I + diag(beta) L (16 x 16 diagonal blocks by substitution, the
//             off-diagonal block by two products) and writes the two operand images the chain
//             reads: B1 = u diag(delta) N_beta^T as a bfloat16 (hi, lo) pair and B2 = -c N_beta^T
//             in tf32 (u, c: the state's deferred scale, below)
//   MMA       (1 warp, one elected lane): every tcgen05.mma, each group's completion by commit
//   chain     (8 warps): the passes over TMEM between the state-dependent products
//   loads     (1 warp): K (64-token tiles) and V (32-token sub-tiles) by TMA, L2 prefetch ahead
//   state     (1 warp): each slot's state into a staging buffer by TMA, S_after out of it
// Per sub-tile j, in tensor-pipe order:
//   E(j)   = V^T B1                      (bf16, issued during the previous sub-tile's pass; N = 64:
//                                         the hi and lo halves land side by side in TMEM)
//   X      = S~ K^T                      (tf32: A = the fp32 state straight from TMEM, K exact)
//   E(j)  += X B2                        (tf32: A = X straight from TMEM, no pass in between)
//   pass   (chain) E = hi half + lo half, split into bfloat16 (hi, lo) A operand
//   S~     = 2^-s S~ + E K               (bf16 (hi, lo) x K; the input state scaled by the
//                                         instruction's power-of-two scale-input-d operand)
// so the chain's own work per sub-tile is one pass over a 128 x 32 block.
//
// Deferred decay.  TMEM holds S~ with the true state S = sig S~.  A sub-tile with decay gamma_C
// takes p = gamma_C sig and a shift s in [0, 15] that brings p 2^s into [1/2, 1) when it can:
// then sig <- p 2^s, u = 1 / sig, c = 2^-s, and MMA_S scales S~ by 2^-s as it accumulates (exact).
// When p < 2^-45 (no shift reaches 2^-30) the chain multiplies S~ by p in a pass instead, sig
// restarts at 1, u = 1 and c = p.  So sig stays in [2^-30, 1] and u below 2^30.  The producer
// and the chain see the same per-sub-tile constants (sig after the sub-tile, the shift, the pass
// factor), which the producer writes beside the images.
//
// Precision.  k, v exact in bfloat16; K K^T exact in fp32.  The state-dependent products read S~
// and X as tf32 (10 explicit mantissa bits, truncated) and B2 is rounded to tf32: errors confined
// to the delta correction.  B1 and E take two-term bfloat16 splits (x = hi + lo, about 2^-16
// relative).  The inverse is formed in fp32.  A CPU model of exactly these roundings gives a state
// error against fp64 of 4.5e-4 at the slowest decay the tests use (4 chunks of 1024 tokens), 5e-6
// at a typical one, and drift numerators within 2.2e-4.
//
// Synchronisation.  Roles hand work to each other through mbarriers only; every wait is bounded
// (about one second, or the workspace header's override); a wait that runs out records
// DELTAS_ERR_TIMEOUT, raises a CTA-wide abort flag so the other roles stop waiting, and the CTA
// drains its MMAs and copies before freeing TMEM.  Heads split between neighbouring CTAs (equal
// tile runs, see ChainSched) hand the state over through the workspace with a bit per CTA boundary
// in the workspace header, which its reader clears after use.
//
// TMEM (512 columns, 128 lanes = d_v): S~ [0,128), S_before [128,256), X [256,288),
// E0 [288,352), E1 [352,416) (each: hi-half product [+0,+32), lo-half product [+32,+64)),
// K K^T [416,480) (lanes 0..63), packed A of MMA_S [480,512) (hi k-step 0, 1, lo k-step 0, 1).
#include <algorithm>
#include <cmath>

#include "internal.cuh"
#include "tc_ptx.cuh"

namespace deltas {
namespace {

using namespace tc;

constexpr int kC = 32;                 // tokens per sub-tile
constexpr int kTile = 64;              // tokens per tile (two sub-tiles; the schedule's unit)
constexpr int kD = 128;                // head dim (d_k = d_v)
constexpr float kHardMin = 0x1p-45f;   // p below this: the state is rescaled by a pass

// ---- roles
constexpr int kChainWarps = 8;
constexpr int kChain = 32 * kChainWarps;
constexpr int kProdWarp0 = 8;          // 8, 9: TMEM readers of producer groups 0, 1; 10, 11: partners
constexpr int kMmaWarp = 12;
constexpr int kLoadWarp = 13;
constexpr int kStateWarp = 14;
constexpr int kThreads = 15 * 32;
constexpr int kBarChain = 1;           // named barriers: chain (256 threads), producer groups (64)
constexpr int kBarProd0 = 2;

// ---- TMEM columns
constexpr uint32_t kTmemCols = 512;
constexpr uint32_t TM_S = 0, TM_SB = 128, TM_X = 256, TM_E = 288, TM_KK = 416, TM_AP = 480;

// ---- shared memory (bytes from a 1024-aligned base)
constexpr uint32_t SM_K = 0;           // 3 tiles x 16 KB: 2 column blocks (d 0-63, 64-127) x 64 rows x 128 B,
                                       // SW128; sub-tile u in rows 32u..32u+31
constexpr uint32_t SM_K32 = 49152;     // 16 KB: one sub-tile's K in fp32, 4 column blocks (32 dims) x 32 rows
                                       // x 128 B, SW128 (the B operand of X); also the K K^T product's
                                       // over-read past the last K tile (rows 64..127 of its M = 128 A)
constexpr uint32_t SM_V = 65536;       // 3 sub-tiles x 8 KB: 2 column blocks x 32 rows x 128 B, SW128
constexpr uint32_t SM_IMG = 90112;     // 4 slots x 12 KB: B1 hi [0, 4 KB) and lo [4, 8 KB) (32 rows x 128 B,
                                       // the first 64 B of a row used), B2 [8, 12 KB) (32 rows x 32 fp32)
constexpr uint32_t kImgSlot = 12288;
constexpr uint32_t SM_SB = 139264;     // 64 KB: state staging, 4 column blocks x 128 rows x 128 B, SW128
constexpr uint32_t SM_PW = 204800;     // producer workspaces, one per group
constexpr int kMS = 36;                // fp32 row stride of M and N (16-byte aligned rows)
constexpr int kPS = 20;                // fp32 row stride of the 16 x 16 product
// beta, delta and (u, c) of the group's sub-tile are double-buffered by tile parity: the partner
// warp writes the next tile's while the other may still read this one's
constexpr int PW_M = 0, PW_N = 32 * kMS, PW_P = 64 * kMS, PW_BETA = PW_P + 16 * kPS, PW_DELTA = PW_BETA + 64,
              PW_UC = PW_DELTA + 64, PW_FLOATS = PW_UC + 8;
constexpr uint32_t kPwBytes = PW_FLOATS * 4;
constexpr uint32_t SM_CONST = SM_PW + 2 * kPwBytes;   // 4 slots x 48 words: per-sub-tile constants
constexpr int kConstWords = 48;        // [0,32) write-size scale per token, 32 sig after, 33 pass factor
                                       // (< 0: none), 34 shift (int)
constexpr uint32_t SM_BYTES = SM_CONST + 4 * kConstWords * 4;
constexpr uint32_t kSmemAlloc = SM_BYTES + 1024;
static_assert(SM_K32 % 1024 == 0 && SM_V % 1024 == 0 && SM_IMG % 1024 == 0 && SM_SB % 1024 == 0 &&
              kImgSlot % 1024 == 0 && SM_PW % 16 == 0 && kPwBytes % 16 == 0, "shared-memory map");
static_assert(SM_IMG == SM_V + 3 * 8192 && SM_SB == SM_IMG + 4 * kImgSlot && SM_PW == SM_SB + 65536, "map order");
static_assert(kSmemAlloc + 1024 <= 232448, "shared memory budget");

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

// (a, b) -> packed bf16 hi = (bf16(a), bf16(b)) and lo = (bf16(a - hi_a), bf16(b - hi_b)), a in the
// low half (even k low: the packing of a TMEM A operand and of a K-major row)
__device__ __forceinline__ void split2(float a, float b, uint32_t& hi, uint32_t& lo) {
    const __nv_bfloat162 hh = __floats2bfloat162_rn(a, b);
    const float2 hf = __bfloat1622float2(hh);
    hi = *reinterpret_cast<const uint32_t*>(&hh);
    lo = pack_bf16x2(a - hf.x, b - hf.y);
}

// fp32 -> tf32 with round-to-nearest (ties away), as the 32-bit container the tensor core reads
__device__ __forceinline__ uint32_t to_tf32(float x) {
    uint32_t y;
    asm("cvt.rna.tf32.f32 %0, %1;" : "=r"(y) : "f"(x));
    return y;
}

// All lanes of a converged warp wait; the result is the same on every lane.
__device__ __forceinline__ bool warp_wait(uint64_t* bar, uint32_t parity, uint64_t budget_ns,
                                          const volatile int* abort) {
    const bool ok = mbar_wait_or_abort(bar, parity, budget_ns, abort);
    return __all_sync(0xffffffffu, ok) != 0;
}

__device__ __forceinline__ void fail(int32_t* status, volatile int* abort, int where) {
    record_status(status, DELTAS_ERR_TIMEOUT, where);
    *abort = 1;
}

// One arrival per warp: every lane's TMEM stores / shared-memory writes were completed and fenced
// before the __syncwarp; lane 0 then arrives (release).
__device__ __forceinline__ void warp_arrive(uint64_t* bar, int lane) {
    __syncwarp();
    if (lane == 0) mbar_arrive(bar);
}

__device__ __forceinline__ int ld_acquire(const uint32_t* p) {
    int v;
    asm volatile("ld.acquire.gpu.global.b32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
    return v;
}
// orders the tensor copies' global accesses with the generic ones around a hand-over bit
__device__ __forceinline__ void fence_proxy_async_global() {
    asm volatile("fence.proxy.async.global;" ::: "memory");
}

// The per-sub-tile decay bookkeeping (see the header): from p = gamma_C sig, the shift s, the
// scale u of the V term, the coefficient c of the X term, the pass factor (< 0: no pass) and sig
// after the sub-tile.
struct DecayStep {
    int shift;
    float u, c, pass, sig;
};
__device__ __forceinline__ DecayStep decay_step(float p) {
    DecayStep d;
    if (!(p >= kHardMin)) {                            // also p = 0 or NaN-free underflow
        d.shift = 0; d.u = 1.f; d.c = p; d.pass = p; d.sig = 1.f;
        return d;
    }
    int e;
    (void)frexpf(p, &e);                               // p = m 2^e, m in [1/2, 1)
    d.shift = min(15, max(0, -e));
    d.sig = ldexpf(p, d.shift);
    d.u = 1.f / d.sig;
    d.c = ldexpf(1.f, -d.shift);
    d.pass = -1.f;
    return d;
}

struct TcArgs {
    int L, Hk, Hv, T, n_tiles;   // n_tiles: 64-token tiles per head
    const float* g;              // [L][T][Hv] log-decay
    const float* beta;           // [L][T][Hv]
    float* state;
    float* partials;
    float* wnorm;
    int32_t* status;
    uint32_t* ho_bits;           // hand-over bits in the workspace header: [0, 16) state, [16, 32) sums
    float* ho_wsum;              // [grid]
    int split;                   // run equal tile runs (ChainSched)
};

// The CTA's work: a sequence of slots, each a run of consecutive tiles of one head.  By default
// the CTA owns heads blockIdx.x, blockIdx.x + gridDim.x, ... whole.  When the heads do not divide
// evenly among the CTAs and the host estimates it faster (a.split), the CTAs instead take equal
// runs of the tile sequence in head order, so that the slowest CTA has one tile more than the
// fastest instead of a whole head more; a head cut by a run boundary is shared by two neighbours.
// CTA i runs the head it shares with CTA i + 1 first (its first tiles; the state at the cut goes
// to hand-over entry i) and the head it shares with CTA i - 1 last (its last tiles, from hand-over
// entry i - 1), so the second part of a shared head is never waited for before its first part is
// long finished.  The split schedule is launched cooperatively, so every CTA is resident.
struct ChainSched {
    int split;
    int pre_lh, pre_len;       // first slot: tiles [0, pre_len) of head pre_lh (none if pre_len == 0)
    int full0, n_full;         // then n_full whole heads from full0 (every gridDim.x-th if !split)
    int suf_lh, suf_from;      // last slot: tiles [suf_from, n) of head suf_lh (none if suf_from == 0)
    int n_slots, NJ;
    __device__ void init(const TcArgs& a) {
        const int n = a.n_tiles, G = (int)gridDim.x, i = (int)blockIdx.x, H = a.L * a.Hv;
        split = a.split && H > G && H % G != 0;
        if (!split) {
            pre_lh = suf_lh = -1; pre_len = suf_from = 0;
            full0 = i; n_full = n_slots = (H - i + G - 1) / G; NJ = n_slots * n;
            return;
        }
        const long long W = (long long)H * n;
        const long long b0 = W * i / G, b1 = W * (i + 1) / G;   // at least n tiles apart (H > G)
        const int hA = (int)(b0 / n), tA = (int)(b0 - (long long)hA * n);
        const int hB = (int)(b1 / n), tB = (int)(b1 - (long long)hB * n);
        suf_lh = hA; suf_from = tA;
        full0 = tA > 0 ? hA + 1 : hA;
        pre_lh = hB; pre_len = tB;
        n_full = hB - full0;
        n_slots = (pre_len > 0 ? 1 : 0) + n_full + (suf_from > 0 ? 1 : 0);
        NJ = (int)(b1 - b0);
    }
    __device__ __forceinline__ bool is_prefix(int k) const { return pre_len > 0 && k == 0; }
    __device__ __forceinline__ bool is_suffix(int k) const { return suf_from > 0 && k == n_slots - 1; }
    __device__ void slot(int k, int n, int& lh, int& tb, int& te) const {
        tb = 0; te = n;
        if (!split) { lh = full0 + k * (int)gridDim.x; return; }
        if (is_prefix(k)) { lh = pre_lh; te = pre_len; return; }
        if (is_suffix(k)) { lh = suf_lh; tb = suf_from; return; }
        lh = full0 + k - (pre_len > 0 ? 1 : 0);
    }
};

// Where a role's current tile lies: slot k, tile jt (of [tb, te)) of head lh = (layer l, value
// head h), key head kh.
struct TileCursor {
    int k, jt, tb, te, lh, l, h, kh;
    __device__ __forceinline__ void set_slot(int slot, const ChainSched& sc, const TcArgs& a) {
        k = slot;
        sc.slot(slot, a.n_tiles, lh, tb, te);
        jt = tb;
        l = lh / a.Hv; h = lh - l * a.Hv;
        kh = (int)(((long long)h * a.Hk) / a.Hv);
    }
    __device__ __forceinline__ void init(const ChainSched& sc, const TcArgs& a) {
        k = -1;
        if (sc.n_slots > 0) set_slot(0, sc, a);
    }
    __device__ __forceinline__ void next(const ChainSched& sc, const TcArgs& a) {
        if (++jt == te && k + 1 < sc.n_slots) set_slot(k + 1, sc, a);
    }
};

// The staging buffer holds a head's [d_v][d_k] fp32 state as four column blocks of 32 floats, each
// 128 rows x 128 bytes with the 128-byte swizzle that TMA writes and reads.  Float offset of 16-byte
// chunk `chunk` (0..31) of row `row`:
__device__ __forceinline__ int sb_idx(int row, int chunk) {
    return (chunk >> 3) * 4096 + row * 32 + (((chunk & 7) ^ (row & 7)) << 2);
}

__global__ void __launch_bounds__(kThreads, 1)
gdn_fused_kernel(const __grid_constant__ CUtensorMap kmap, const __grid_constant__ CUtensorMap vmap,
                 const __grid_constant__ CUtensorMap smap, const __grid_constant__ CUtensorMap hmap,
                 TcArgs a)
{
    extern __shared__ uint8_t smem_raw[];
    uint8_t* sm = smem_raw + ((1024 - (smem_u32(smem_raw) & 1023)) & 1023);
    // loads -> roles: K tiles, V sub-tiles full; MMA -> loader: their empties.  producer <-> MMA:
    // operand images full / empty (the chain's constants read too), K K^T done / read.  state
    // staging full (mb_st) and released by the chain (mb_sfree).  MMA -> chain: u (E ready), s
    // (state updated); chain -> MMA: sready (state and K in fp32 ready for X), uready (A packed).
    __shared__ uint64_t mb_kfull[3], mb_kempty[3], mb_vfull[3], mb_vempty[3], mb_ifull[4], mb_iempty[4];
    __shared__ uint64_t mb_kk, mb_kkfree, mb_st, mb_sfree, mb_sready, mb_x, mb_u, mb_uready, mb_s, mb_fin;
    __shared__ uint32_t s_tmem;
    __shared__ int s_abort;
    __shared__ float s_red[2][kChainWarps];
    __shared__ float s_u2[2][kC];                     // per-token squared write sizes (sub-tile parity)
    volatile int* abort_flag = &s_abort;

    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    // bounded-wait budget: the workspace header's override (microseconds) or about one second
    const uint32_t budget_us = reinterpret_cast<const volatile uint32_t*>(a.status)[2];
    const uint64_t budget = budget_us ? (uint64_t)budget_us * 1000ull : kWaitBudgetNs;
    ChainSched sch;
    sch.init(a);
    const int n_slots = sch.n_slots;
    const int NJ = sch.NJ;                            // tiles of this CTA
    const int NS = 2 * NJ;                            // sub-tiles
    const int me = (int)blockIdx.x;
    uint32_t* bits_state = a.ho_bits;
    uint32_t* bits_wsum = a.ho_bits + 16;

    if (warp == kMmaWarp) {
        tmem_alloc(&s_tmem, kTmemCols);
        tmem_relinquish();
        if (lane == 0) {
            for (int b = 0; b < 3; ++b) {
                mbar_init(&mb_kfull[b], 1); mbar_init(&mb_kempty[b], 1);
                mbar_init(&mb_vfull[b], 1); mbar_init(&mb_vempty[b], 1);
            }
            for (int b = 0; b < 4; ++b) { mbar_init(&mb_ifull[b], 2); mbar_init(&mb_iempty[b], 1 + kChainWarps); }
            mbar_init(&mb_kk, 1); mbar_init(&mb_kkfree, 2);
            mbar_init(&mb_st, 1); mbar_init(&mb_sfree, kChainWarps);
            mbar_init(&mb_sready, kChainWarps); mbar_init(&mb_x, 1); mbar_init(&mb_u, 1);
            mbar_init(&mb_uready, kChainWarps);
            mbar_init(&mb_s, 1); mbar_init(&mb_fin, 1);
            fence_barrier_init();
        }
    }
    if (warp == kLoadWarp && lane == 0) { prefetch_tensormap(&kmap); prefetch_tensormap(&vmap); }
    if (warp == kStateWarp && lane == 0) { prefetch_tensormap(&smap); prefetch_tensormap(&hmap); }
    if (tid == 0) s_abort = 0;
    if (tid < 2 * kC) s_u2[tid >> 5][tid & (kC - 1)] = 0.f;
    grid_dep_launch();                                // the next kernel (the score) may be scheduled
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tm = s_tmem;
    const float* cst = reinterpret_cast<const float*>(sm + SM_CONST);

    if (warp == kMmaWarp) {
        // =========================================================== MMA issue (converged warp;
        // one elected lane issues each group and commits it)
        const uint32_t idX = idesc_tf32(128, 32);
        const uint32_t idE = idesc_bf16(128, 64, 1, 0);
        const uint32_t idS = idesc_bf16(128, 128, 0, 1);
        const uint32_t idK = idesc_bf16(128, 64, 0, 0);
        // K K^T of tile J (M = 128: rows 64..127 of A read the 16 KB past the tile; their output
        // lanes are ignored).  Waits for the tile and for both producer groups to have read the
        // previous product out of TMEM.
        auto issue_kk = [&](int J) -> bool {
            const uint32_t base = smem_u32(sm + SM_K + (J % 3) * 16384);
            uint64_t d[2][4];
#pragma unroll
            for (int s = 0; s < 8; ++s) {
                d[s >> 2][s & 3] = sdesc_sw128(base + (s >> 2) * 8192 + (s & 3) * 32, 16, 1024);
                pin(d[s >> 2][s & 3]);
            }
            if (!warp_wait(&mb_kfull[J % 3], (J / 3) & 1, budget, abort_flag)) return false;
            if (J > 0 && !warp_wait(&mb_kkfree, (J - 1) & 1, budget, abort_flag)) return false;
            tc_fence_after();
            if (elect_one()) {
                mma4_bf16_ss_1t(tm + TM_KK, d[0], d[0], idK, 0);
                mma4_bf16_ss_1t(tm + TM_KK, d[1], d[1], idK, 1);
            }
            __syncwarp();
            mma_commit(&mb_kk);
            return true;
        };
        // E(j) <- V(j)^T B1(j): A = the V sub-tile read MN-major, B = the 64-row (hi, lo) image
        auto issue_einit = [&](int j) -> bool {
            const uint32_t vb = smem_u32(sm + SM_V + (j % 3) * 8192);
            const uint32_t ib = smem_u32(sm + SM_IMG + (j & 3) * kImgSlot);
            const uint64_t a0 = sdesc_sw128(vb, 4096, 1024), a1 = sdesc_sw128(vb + 2048, 4096, 1024);
            const uint64_t b0 = sdesc_sw128(ib, 16, 1024), b1 = sdesc_sw128(ib + 32, 16, 1024);
            pin(a0); pin(a1); pin(b0); pin(b1);
            if (!warp_wait(&mb_vfull[j % 3], (j / 3) & 1, budget, abort_flag)) return false;
            if (!warp_wait(&mb_ifull[j & 3], (j >> 2) & 1, budget, abort_flag)) return false;
            tc_fence_after();
            if (elect_one()) {
                mma_bf16_1t(tm + TM_E + (j & 1) * 64, a0, b0, idE, 0);
                mma_bf16_1t(tm + TM_E + (j & 1) * 64, a1, b1, idE, 1);
            }
            __syncwarp();
            mma_commit(&mb_vempty[j % 3]);
            return true;
        };
        bool ok = true;
        if (NS > 0) {
            ok = issue_kk(0);
            if (ok && NJ > 1) ok = issue_kk(1);
            if (ok) ok = issue_einit(0);            // completes before X(0)'s commit
            if (!ok) fail(a.status, abort_flag, 1);
        }
        // The tensor core does not order an MMA that reads a TMEM region as its A operand after an
        // earlier MMA that wrote it (measured: X read by the next product lacked the last of its 16
        // k-steps), so each such hand-off waits for the writer's commit: X before E += X B2, and
        // the updated state before the next X.  Independent work fills the turnarounds: the next
        // sub-tile's E product between X and E += X B2, the K K^T product during the chain's pass.
        for (int j = 0; ok && j < NS; ++j) {
            const uint32_t eb = tm + TM_E + (j & 1) * 64;
            int shift = 0;
            {   // X <- S~ K^T (A: the state from TMEM as tf32, 8 columns per K = 8 step; B: K in fp32)
                uint32_t ax[4][4];
                uint64_t bx[4][4];
                const uint32_t k32 = smem_u32(sm + SM_K32);
#pragma unroll
                for (int s = 0; s < 16; ++s) {
                    ax[s >> 2][s & 3] = tm + TM_S + 8 * s;
                    bx[s >> 2][s & 3] = sdesc_sw128(k32 + (s >> 2) * 4096 + (s & 3) * 32, 16, 1024);
                    pin(ax[s >> 2][s & 3]); pin(bx[s >> 2][s & 3]);
                }
                if (!warp_wait(&mb_sready, j & 1, budget, abort_flag)) { fail(a.status, abort_flag, 2); break; }
                if (j > 0 && !warp_wait(&mb_s, (j - 1) & 1, budget, abort_flag)) { fail(a.status, abort_flag, 7); break; }
                if (!warp_wait(&mb_ifull[j & 3], (j >> 2) & 1, budget, abort_flag)) { fail(a.status, abort_flag, 3); break; }
                // read while the image slot is held (released once its products and the chain are done)
                shift = reinterpret_cast<const volatile int*>(cst + (j & 3) * kConstWords)[34];
                tc_fence_after();
                if (elect_one()) {
#pragma unroll
                    for (int g4 = 0; g4 < 4; ++g4) mma4_tf32_ta_1t(tm + TM_X, ax[g4], bx[g4], idX, g4 != 0);
                }
                __syncwarp();
                mma_commit(&mb_x);
            }
            if (j + 1 < NS && !issue_einit(j + 1)) { fail(a.status, abort_flag, 5); break; }
            {   // E(j) += X B2 (A: X from TMEM as tf32); E(j)'s own product completed before X's commit
                uint32_t au[4];
                uint64_t bu[4];
                const uint32_t b2 = smem_u32(sm + SM_IMG + (j & 3) * kImgSlot + 8192);
#pragma unroll
                for (int s = 0; s < 4; ++s) {
                    au[s] = tm + TM_X + 8 * s;
                    bu[s] = sdesc_sw128(b2 + 32 * s, 16, 1024);
                    pin(au[s]); pin(bu[s]);
                }
                if (!warp_wait(&mb_x, j & 1, budget, abort_flag)) { fail(a.status, abort_flag, 8); break; }
                tc_fence_after();
                if (elect_one()) mma4_tf32_ta_1t(eb, au, bu, idX, 1);
                __syncwarp();
                mma_commit(&mb_u);
                mma_commit(&mb_iempty[j & 3]);
            }
            // K K^T one and a half tiles ahead of the chain, while the chain runs its pass
            if ((j & 1) && (j + 3) / 2 < NJ && !issue_kk((j + 3) / 2)) { fail(a.status, abort_flag, 4); break; }
            {   // S~ = 2^-shift S~ + E K  (A: E hi / lo packed in TMEM; K read MN-major)
                uint32_t as_[4];
                uint64_t bs[4];
                const uint32_t kb = smem_u32(sm + SM_K + ((j >> 1) % 3) * 16384) + (j & 1) * 4096;
#pragma unroll
                for (int s = 0; s < 4; ++s) {
                    as_[s] = tm + TM_AP + 8 * s;
                    bs[s] = sdesc_sw128(kb + (s & 1) * 2048, 8192, 1024);
                    pin(as_[s]); pin(bs[s]);
                }
                if (!warp_wait(&mb_uready, j & 1, budget, abort_flag)) { fail(a.status, abort_flag, 6); break; }
                tc_fence_after();
                if (elect_one()) mma4_bf16_ta_shift_1t(shift, tm + TM_S, as_, bs, idS);
                __syncwarp();
                mma_commit(&mb_s);
                if (j & 1) mma_commit(&mb_kempty[(j >> 1) % 3]);   // the tile's last reader
            }
        }
        if (__any_sync(0xffffffffu, *abort_flag != 0)) {
            mma_commit(&mb_fin);                       // every MMA this warp issued has completed
            mbar_wait(&mb_fin, 0, budget);
        }
        __syncwarp();
    } else if (warp == kLoadWarp) {
        // =========================================================== K tiles and V sub-tiles in
        // order, each into its buffer once the MMA that last read the buffer has completed; the
        // tiles three ahead are prefetched into L2
        TileCursor cc, pf;
        cc.init(sch, a);
        pf.init(sch, a);
        int kp[3] = {-1, -1, -1}, vp[3] = {-1, -1, -1};   // last tile / sub-tile loaded per buffer
        grid_dep_wait();
        // prime the prefetch cursor three tiles ahead
        for (int i = 0; i < 3 && i < NJ; ++i) {
            if (elect_one()) {
                tma_prefetch_4d(&kmap, 0, pf.kh, pf.jt * kTile, pf.l);
                tma_prefetch_4d(&kmap, 64, pf.kh, pf.jt * kTile, pf.l);
                tma_prefetch_4d(&vmap, 0, pf.h, pf.jt * kTile, pf.l);
                tma_prefetch_4d(&vmap, 64, pf.h, pf.jt * kTile, pf.l);
                tma_prefetch_4d(&vmap, 0, pf.h, pf.jt * kTile + kC, pf.l);
                tma_prefetch_4d(&vmap, 64, pf.h, pf.jt * kTile + kC, pf.l);
            }
            __syncwarp();
            pf.next(sch, a);
        }
        bool ok = true;
        for (int J = 0; ok && J < NJ; ++J) {
            if (J + 3 < NJ) {
                if (elect_one()) {
                    tma_prefetch_4d(&kmap, 0, pf.kh, pf.jt * kTile, pf.l);
                    tma_prefetch_4d(&kmap, 64, pf.kh, pf.jt * kTile, pf.l);
                    tma_prefetch_4d(&vmap, 0, pf.h, pf.jt * kTile, pf.l);
                    tma_prefetch_4d(&vmap, 64, pf.h, pf.jt * kTile, pf.l);
                    tma_prefetch_4d(&vmap, 0, pf.h, pf.jt * kTile + kC, pf.l);
                    tma_prefetch_4d(&vmap, 64, pf.h, pf.jt * kTile + kC, pf.l);
                }
                __syncwarp();
                pf.next(sch, a);
            }
            const int bk = J % 3;
            if (J >= 3 && !warp_wait(&mb_kempty[bk], ((J / 3) - 1) & 1, budget, abort_flag)) { fail(a.status, abort_flag, 30); break; }
            if (elect_one()) {
                uint8_t* dst = sm + SM_K + bk * 16384;
                mbar_arrive_expect_tx(&mb_kfull[bk], 16384);
                tma_load_4d(dst, &kmap, &mb_kfull[bk], 0, cc.kh, cc.jt * kTile, cc.l);
                tma_load_4d(dst + 8192, &kmap, &mb_kfull[bk], 64, cc.kh, cc.jt * kTile, cc.l);
            }
            __syncwarp();
            kp[bk] = J;
            for (int u = 0; u < 2; ++u) {
                const int j = 2 * J + u, bv = j % 3;
                if (j >= 3 && !warp_wait(&mb_vempty[bv], ((j / 3) - 1) & 1, budget, abort_flag)) {
                    fail(a.status, abort_flag, 31);
                    ok = false;
                    break;
                }
                if (elect_one()) {
                    uint8_t* dst = sm + SM_V + bv * 8192;
                    mbar_arrive_expect_tx(&mb_vfull[bv], 8192);
                    tma_load_4d(dst, &vmap, &mb_vfull[bv], 0, cc.h, cc.jt * kTile + kC * u, cc.l);
                    tma_load_4d(dst + 4096, &vmap, &mb_vfull[bv], 64, cc.h, cc.jt * kTile + kC * u, cc.l);
                }
                __syncwarp();
                vp[bv] = j;
            }
            cc.next(sch, a);
        }
        if (__any_sync(0xffffffffu, *abort_flag != 0) && lane == 0) {
            // every copy this warp issued lands before the CTA ends
            for (int b = 0; b < 3; ++b) {
                if (kp[b] >= 0) mbar_wait(&mb_kfull[b], (kp[b] / 3) & 1, budget);
                if (vp[b] >= 0) mbar_wait(&mb_vfull[b], (vp[b] / 3) & 1, budget);
            }
        }
        __syncwarp();
    } else if (warp == kStateWarp) {
        // =========================================================== state moves (lane 0).  Phases
        // of mb_st: 0 = the first slot's state staged; k + 1 = what the boundary after slot k
        // needs: the state of slot k + 1, or after the last slot a free buffer (when the last slot
        // ends a head begun by CTA i - 1: that head's state before the chunk, for its drift).
        // Phases of mb_sfree: 0 = the first state is in TMEM; k + 1 = slot k's final state is
        // staged.  A first slot that begins a head shared with CTA i + 1 leaves its state in
        // hand-over entry i; a last slot that ends a head shared with CTA i - 1 starts from entry
        // i - 1 once that entry's bit is set (bounded wait), and clears the bit.
        if (lane == 0 && n_slots > 0) {
            float* sbuf = reinterpret_cast<float*>(sm + SM_SB);
            int loads = 0, seen = 0;                   // copies into the staging buffer issued / landed
            auto load_rows = [&](const CUtensorMap* map, int row) {
                mbar_arrive_expect_tx(&mb_st, kD * kD * 4);
#pragma unroll
                for (int b = 0; b < 4; ++b) tma_load_2d(sbuf + 4096 * b, map, &mb_st, 32 * b, row);
                ++loads;
            };
            auto load_state = [&](int slot) -> bool {
                int lh, tb, te;
                sch.slot(slot, a.n_tiles, lh, tb, te);
                if (!sch.is_suffix(slot)) { load_rows(&smap, lh * kD); return true; }
                const uint32_t bit = 1u << ((me - 1) & 31);
                uint32_t* w = bits_state + ((me - 1) >> 5);
                const uint64_t t0 = global_ns();
                while ((ld_acquire(w) & bit) == 0) {
                    if (*abort_flag || global_ns() - t0 > budget) return false;
                    __nanosleep(64);
                }
                atomicAnd(w, ~bit);                    // consumed: zero for the next call
                fence_proxy_async_global();
                load_rows(&hmap, (me - 1) * kD);
                return true;
            };
            auto final_phase = [&]() {                 // what the boundary after the last slot reads
                if (sch.is_suffix(n_slots - 1)) load_rows(&smap, sch.suf_lh * kD);
                else mbar_arrive(&mb_st);
            };
            grid_dep_wait();
            bool ok = load_state(0);
            if (!ok) fail(a.status, abort_flag, 42);
            if (ok) {
                ok = mbar_wait_or_abort(&mb_sfree, 0, budget, abort_flag);
                if (!ok) fail(a.status, abort_flag, 40);
            }
            seen = loads;                              // the chain has consumed it
            if (ok) {
                if (n_slots > 1) {
                    ok = load_state(1);
                    if (!ok) fail(a.status, abort_flag, 43);
                } else {
                    final_phase();
                }
            }
            for (int k = 0; ok && k < n_slots; ++k) {
                if (!mbar_wait_or_abort(&mb_sfree, (k + 1) & 1, budget, abort_flag)) { fail(a.status, abort_flag, 41); break; }
                seen = loads;
                int lh, tb, te;
                sch.slot(k, a.n_tiles, lh, tb, te);
                const bool hand_over = sch.is_prefix(k);
                const CUtensorMap* dst = hand_over ? &hmap : &smap;
                const int row = (hand_over ? me : lh) * kD;
#pragma unroll
                for (int b = 0; b < 4; ++b) tma_store_2d(dst, sbuf + 4096 * b, 32 * b, row);
                bulk_commit();
                if (hand_over) {
                    bulk_wait0();                      // the state is in global memory ...
                    fence_proxy_async_global();
                    __threadfence();
                    atomicOr(bits_state + (me >> 5), 1u << (me & 31));   // ... before CTA i + 1 reads it
                }
                if (k + 2 <= n_slots) {
                    bulk_wait_read0();                 // slot k's state has left the buffer
                    if (k + 2 < n_slots) {
                        if (!load_state(k + 2)) { fail(a.status, abort_flag, 43); break; }
                    } else {
                        final_phase();
                    }
                }
            }
            bulk_wait0();                              // every state store is complete
            if (loads > seen) mbar_wait(&mb_st, (loads - 1) & 1, budget);   // abort: a load in flight
        }
        __syncwarp();
    } else if (warp >= kProdWarp0) {
        // =========================================================== producer: operand images of
        // the sub-tiles of parity G, and the per-sub-tile decay constants
        const int G = (warp - kProdWarp0) & 1;
        const bool tm_warp = warp < kProdWarp0 + 2;    // reads TMEM lanes 32 G .. 32 G + 31
        const int gt = (tm_warp ? 0 : 32) + lane;      // thread of the group, 0..63
        float* pw = reinterpret_cast<float*>(sm + SM_PW + G * kPwBytes);
        float* Mm = pw + PW_M;                         // diag(beta) L of the sub-tile, rows of kMS
        float* Nm = pw + PW_N;                         // (I + diag(beta) L)^-1
        float* Pm = pw + PW_P;                         // 16 x 16 product of the off-diagonal block
        float* sBeta0 = pw + PW_BETA;                  // [2][32]
        float* sDelta0 = pw + PW_DELTA;                // [2][32]
        float* sUC0 = pw + PW_UC;                      // [2][u, c, -, -]
        const int bar_id = kBarProd0 + G;
        TileCursor cc;
        cc.init(sch, a);
        // g of tokens lane and 32 + lane of the tile, beta of this group's token lane (partner warp),
        // loaded one tile ahead of use
        float pg0 = 0.f, pg1 = 0.f, pb = 0.f;
        auto load_gb = [&](const TileCursor& c) {
            const int t0 = c.jt * kTile + lane, t1 = t0 + kC, tg = G ? t1 : t0;
            const size_t base = (size_t)c.l * a.T;
            pg0 = t0 < a.T ? a.g[(base + t0) * a.Hv + c.h] : 0.f;
            pg1 = t1 < a.T ? a.g[(base + t1) * a.Hv + c.h] : 0.f;
            pb = tg < a.T ? a.beta[(base + tg) * a.Hv + c.h] : 0.f;
        };
        if (!tm_warp && NJ > 0) { grid_dep_wait(); load_gb(cc); }
        float sig = 1.f;
        int prev_slot = -1;
        bool failed = false;
        for (int J = 0; J < NJ; ++J) {
            const int j = 2 * J + G;
            float* sBeta = sBeta0 + 32 * (J & 1);
            float* sDelta = sDelta0 + 32 * (J & 1);
            float* sUC = sUC0 + 4 * (J & 1);
            float kk[32];
            DecayStep dmine;
            float wn = 0.f;
            if (!tm_warp) {
                const float g0 = pg0, g1 = pg1, bt = pb;
                if (J + 1 < NJ) {                       // the next tile's g, beta
                    TileCursor nx = cc;
                    nx.next(sch, a);
                    load_gb(nx);
                }
                if (cc.k != prev_slot) sig = 1.f;       // a slot starts from the true state
                prev_slot = cc.k;
                float G0 = g0, G1 = g1;                 // inclusive scans over the two sub-tiles
#pragma unroll
                for (int m = 1; m < 32; m <<= 1) {
                    const float y0 = __shfl_up_sync(0xffffffffu, G0, m);
                    const float y1 = __shfl_up_sync(0xffffffffu, G1, m);
                    if (lane >= m) { G0 += y0; G1 += y1; }
                }
                const float GC0 = __shfl_sync(0xffffffffu, G0, 31), GC1 = __shfl_sync(0xffffffffu, G1, 31);
                const DecayStep d0 = decay_step(expf(GC0) * sig);
                const DecayStep d1 = decay_step(expf(GC1) * d0.sig);
                sig = d1.sig;
                dmine = G ? d1 : d0;
                const float Gm = G ? G1 : G0, GCm = G ? GC1 : GC0;
                const float delta = expf(GCm - Gm);
                sBeta[lane] = bt;
                sDelta[lane] = delta;
                const float ud = dmine.u * delta;
                wn = ud >= 0x1p-60f ? 1.f / ud : 0.f;   // column t of E is u delta_t u_t
                if (lane == 0) { sUC[0] = dmine.u; sUC[1] = dmine.c; }
            } else {
                const bool ok = mbar_wait_or_abort(&mb_kk, J & 1, budget, abort_flag);
                if (!ok) { fail(a.status, abort_flag, 20); failed = true; }
                tc_fence_after();
                if (ok) {
                    tmem_ld32(tm + ((uint32_t)(32 * G) << 16) + TM_KK + 32 * G, kk);
                    tmem_ld_wait();
                }
                tc_fence_before();
                __syncwarp();
                if (lane == 0) mbar_arrive(&mb_kkfree);
            }
            if (named_sync_or(bar_id, 64, failed || *abort_flag)) break;     // (1)
            if (tm_warp) {                              // row t of diag(beta) L: beta_t k_t.k_c, c < t
                const float bt = sBeta[lane];
                float* row = Mm + lane * kMS;
#pragma unroll
                for (int c4 = 0; c4 < 8; ++c4) {
                    float4 v;
                    v.x = (4 * c4 + 0 < lane) ? bt * kk[4 * c4 + 0] : 0.f;
                    v.y = (4 * c4 + 1 < lane) ? bt * kk[4 * c4 + 1] : 0.f;
                    v.z = (4 * c4 + 2 < lane) ? bt * kk[4 * c4 + 2] : 0.f;
                    v.w = (4 * c4 + 3 < lane) ? bt * kk[4 * c4 + 3] : 0.f;
                    *reinterpret_cast<float4*>(row + 4 * c4) = v;
                }
            }
            if (named_sync_or(bar_id, 64, *abort_flag)) break;               // (2)
            if (tm_warp) {
                // the two 16 x 16 diagonal blocks of N by forward substitution, one column per lane
                const int b = lane >> 4, jc = lane & 15, o = 16 * b;
                float x[16];
#pragma unroll
                for (int rr = 0; rr < 16; ++rr) x[rr] = (rr == jc) ? 1.f : 0.f;
#pragma unroll
                for (int rr = 1; rr < 16; ++rr) {
                    const float* mr = Mm + (o + rr) * kMS + o;
                    float s0 = 0.f, s1 = 0.f;
#pragma unroll
                    for (int c = 0; c < rr; c += 4) {
                        const float4 v = *reinterpret_cast<const float4*>(mr + c);
                        s0 = fmaf(v.x, x[c], s0);
                        if (c + 1 < rr) s1 = fmaf(v.y, x[c + 1], s1);
                        if (c + 2 < rr) s0 = fmaf(v.z, x[c + 2], s0);
                        if (c + 3 < rr) s1 = fmaf(v.w, x[c + 3], s1);
                    }
                    if (rr > jc) x[rr] = -(s0 + s1);
                }
#pragma unroll
                for (int rr = 0; rr < 16; ++rr) Nm[(o + rr) * kMS + o + jc] = x[rr];
                if (b == 0) {
#pragma unroll
                    for (int rr = 0; rr < 16; ++rr) Nm[rr * kMS + 16 + jc] = 0.f;   // upper block
                }
            }
            if (named_sync_or(bar_id, 64, *abort_flag)) break;               // (3)
            {   // P = M10 N00, then N10 = -N11 P (16 x 16 blocks; 4 outputs per thread)
                const int r = gt >> 2, c0 = 4 * (gt & 3);
                float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
                const float* mrow = Mm + (16 + r) * kMS;
#pragma unroll
                for (int a4 = 0; a4 < 16; a4 += 4) {
                    const float4 mv = *reinterpret_cast<const float4*>(mrow + a4);
                    const float m4[4] = {mv.x, mv.y, mv.z, mv.w};
#pragma unroll
                    for (int e = 0; e < 4; ++e) {
                        const float4 nv = *reinterpret_cast<const float4*>(Nm + (a4 + e) * kMS + c0);
                        acc.x = fmaf(m4[e], nv.x, acc.x); acc.y = fmaf(m4[e], nv.y, acc.y);
                        acc.z = fmaf(m4[e], nv.z, acc.z); acc.w = fmaf(m4[e], nv.w, acc.w);
                    }
                }
                *reinterpret_cast<float4*>(Pm + r * kPS + c0) = acc;
                if (named_sync_or(bar_id, 64, *abort_flag)) break;           // (4)
                acc = make_float4(0.f, 0.f, 0.f, 0.f);
                const float* nrow = Nm + (16 + r) * kMS + 16;
#pragma unroll
                for (int a4 = 0; a4 < 16; a4 += 4) {
                    const float4 nv = *reinterpret_cast<const float4*>(nrow + a4);
                    const float n4[4] = {nv.x, nv.y, nv.z, nv.w};
#pragma unroll
                    for (int e = 0; e < 4; ++e) {
                        const float4 pv = *reinterpret_cast<const float4*>(Pm + (a4 + e) * kPS + c0);
                        acc.x = fmaf(n4[e], pv.x, acc.x); acc.y = fmaf(n4[e], pv.y, acc.y);
                        acc.z = fmaf(n4[e], pv.z, acc.z); acc.w = fmaf(n4[e], pv.w, acc.w);
                    }
                }
                *reinterpret_cast<float4*>(Nm + (16 + r) * kMS + c0) = make_float4(-acc.x, -acc.y, -acc.z, -acc.w);
            }
            if (named_sync_or(bar_id, 64, *abort_flag)) break;               // (5)
            // the image slot is free once sub-tile j - 4's products and the chain have read it
            if (j >= 4) {
                const bool ok = mbar_wait_or_abort(&mb_iempty[j & 3], ((j >> 2) - 1) & 1, budget, abort_flag);
                if (!ok) { fail(a.status, abort_flag, 21); failed = true; }
            }
            if (named_sync_or(bar_id, 64, failed || *abort_flag)) break;     // (6)
            {   // images: row t = gt / 2, columns 16 hc .. 16 hc + 15 of N_beta = N diag(beta)
                const int t = gt >> 1, hc = gt & 1;
                const float u = sUC[0], cX = sUC[1];
                uint8_t* slot = sm + SM_IMG + (j & 3) * kImgSlot;
                float nb[16], w1[16];
#pragma unroll
                for (int e = 0; e < 4; ++e) {
                    const float4 nv = *reinterpret_cast<const float4*>(Nm + t * kMS + 16 * hc + 4 * e);
                    const float4 bv = *reinterpret_cast<const float4*>(sBeta + 16 * hc + 4 * e);
                    const float4 dv = *reinterpret_cast<const float4*>(sDelta + 16 * hc + 4 * e);
                    nb[4 * e] = nv.x * bv.x; nb[4 * e + 1] = nv.y * bv.y;
                    nb[4 * e + 2] = nv.z * bv.z; nb[4 * e + 3] = nv.w * bv.w;
                    w1[4 * e] = u * nb[4 * e] * dv.x; w1[4 * e + 1] = u * nb[4 * e + 1] * dv.y;
                    w1[4 * e + 2] = u * nb[4 * e + 2] * dv.z; w1[4 * e + 3] = u * nb[4 * e + 3] * dv.w;
                }
#pragma unroll
                for (int e = 0; e < 4; ++e) {          // B2 = -c N_beta, tf32, row t chunks 4 hc + e
                    const uint4 w = make_uint4(to_tf32(-cX * nb[4 * e]), to_tf32(-cX * nb[4 * e + 1]),
                                               to_tf32(-cX * nb[4 * e + 2]), to_tf32(-cX * nb[4 * e + 3]));
                    *reinterpret_cast<uint4*>(slot + 8192 + sw128_offset(t, 4 * hc + e)) = w;
                }
#pragma unroll
                for (int e = 0; e < 2; ++e) {          // B1 = u N_beta diag(delta), (hi, lo)
                    uint32_t h[4], l[4];
#pragma unroll
                    for (int i = 0; i < 4; ++i) split2(w1[8 * e + 2 * i], w1[8 * e + 2 * i + 1], h[i], l[i]);
                    *reinterpret_cast<uint4*>(slot + sw128_offset(t, 2 * hc + e)) = make_uint4(h[0], h[1], h[2], h[3]);
                    *reinterpret_cast<uint4*>(slot + 4096 + sw128_offset(t, 2 * hc + e)) = make_uint4(l[0], l[1], l[2], l[3]);
                }
            }
            if (!tm_warp) {                             // the chain's and the MMA's constants
                float* cs = const_cast<float*>(cst) + (j & 3) * kConstWords;
                cs[lane] = wn;
                if (lane == 0) {
                    cs[32] = dmine.sig;
                    cs[33] = dmine.pass;
                    reinterpret_cast<int*>(cs)[34] = dmine.shift;
                }
            }
            fence_async_smem();                         // generic writes -> the tensor core's reads
            __syncwarp();
            if (lane == 0) mbar_arrive(&mb_ifull[j & 3]);
            cc.next(sch, a);
        }
    } else {
        // =========================================================== state chain (warps 0-7)
        const int q = warp & 3, hh = warp >> 2;          // TMEM lane quadrant, column half
        const int r = 32 * q + lane;                     // row of S (value index)
        const uint32_t lane_off = (uint32_t)(32 * q) << 16;
        float* sbuf = reinterpret_cast<float*>(sm + SM_SB);   // swizzled rows, see sb_idx
        int st_seen = 0;                                 // mb_st phases waited for (uniform)
        TileCursor cc;
        cc.init(sch, a);
        // K of sub-tile jj (TMA tile, rows 32 (jj & 1) ..) in fp32 (exact, and exact in tf32) into
        // the B operand buffer of X.  Called between MMA_X(jj-1), the last reader of the buffer, and
        // the ready signal of sub-tile jj.
        auto make_k32 = [&](int jj) -> bool {
            const int bk = (jj >> 1) % 3;
            const bool ok = mbar_wait_or_abort(&mb_kfull[bk], ((jj >> 1) / 3) & 1, budget, abort_flag);
            const uint8_t* kb = sm + SM_K + bk * 16384;
            const int r0 = 32 * (jj & 1);
#pragma unroll
            for (int u = 0; u < 2; ++u) {                  // 32 rows x 16 chunks of 8 bf16
                const int e = tid + kChain * u;
                const int t = e >> 4, c16 = e & 15, cb = c16 >> 3, c = c16 & 7;
                const uint4 w = *reinterpret_cast<const uint4*>(kb + cb * 8192 + sw128_offset(r0 + t, c));
                const uint32_t wv[4] = {w.x, w.y, w.z, w.w};
                uint32_t f[8];
#pragma unroll
                for (int i = 0; i < 4; ++i) {
                    f[2 * i] = wv[i] << 16;
                    f[2 * i + 1] = wv[i] & 0xFFFF0000u;
                }
                // dims 64 cb + 8 c .. + 7: fp32 block 2 cb + c / 4, chunks 2 (c % 4) and 2 (c % 4) + 1
                uint8_t* rowp = sm + SM_K32 + (2 * cb + (c >> 2)) * 4096;
                const int q0 = 2 * (c & 3);
                *reinterpret_cast<uint4*>(rowp + sw128_offset(t, q0)) = make_uint4(f[0], f[1], f[2], f[3]);
                *reinterpret_cast<uint4*>(rowp + sw128_offset(t, q0 + 1)) = make_uint4(f[4], f[5], f[6], f[7]);
            }
            fence_async_smem();                            // generic writes -> the tensor core's reads
            return ok;
        };
        float den = 0.f, sig = 1.f;
        // Write sizes (optional): column t of E is u delta_t u_t, u_t = beta_t (v_t - alpha_t S_{t-1}
        // k_t) the token's write.  The pass sums each column's squares over the warp's 32 rows,
        // rescales them by the constant (1 / (u delta_t))^2 and adds them into s_u2 (four warps per
        // column); at the next sub-tile warp 0 takes the square roots and sums them into the head's
        // total.
        const bool want_w = a.wnorm != nullptr;
        float wacc = 0.f;                                  // warp 0: the slot's running sum
        int prev_lh = -1, prev_slot = -1;
        bool prev_last = false;
        // a head's write-size sum: to hand-over entry i when the slot begins a head shared with
        // CTA i + 1, else (with the first part's sum from entry i - 1 when it ends a head shared
        // with CTA i - 1) to the output; warp 0, lane 0
        auto put_wsum = [&](int slot, int lh, float sum) -> bool {
            if (sch.is_prefix(slot)) {
                a.ho_wsum[me] = sum;
                __threadfence();
                atomicOr(bits_wsum + (me >> 5), 1u << (me & 31));
                return true;
            }
            if (sch.is_suffix(slot)) {
                const uint32_t bit = 1u << ((me - 1) & 31);
                uint32_t* w = bits_wsum + ((me - 1) >> 5);
                const uint64_t t0 = global_ns();
                while ((ld_acquire(w) & bit) == 0) {
                    if (*abort_flag || global_ns() - t0 > budget) return false;
                    __nanosleep(64);
                }
                sum += *reinterpret_cast<volatile const float*>(a.ho_wsum + me - 1);
                atomicAnd(w, ~bit);
            }
            a.wnorm[lh] = sum;
            return true;
        };
        auto fold_writes = [&](int jj) {                   // warp 0: sub-tile jj's sizes into wacc
            float* b = s_u2[jj & 1];
            float sacc = sqrtf(b[lane]);
            b[lane] = 0.f;
#pragma unroll
            for (int m = 16; m >= 1; m >>= 1) sacc += __shfl_xor_sync(0xffffffffu, sacc, m);
            wacc += sacc;
        };
        bool stop = false;
        for (int J = 0; J < NJ && !stop; ++J) {
            for (int u = 0; u < 2; ++u) {
                const int j = 2 * J + u;
                const int lh = cc.lh, slot = cc.k;
                const bool last = u == 1 && cc.jt == cc.te - 1;   // the slot's last sub-tile
                if (named_sync_or(kBarChain, kChain, *abort_flag)) { stop = true; break; }
                if (want_w && j > 0 && warp == 0) {
                    fold_writes(j - 1);
                    if (prev_last) {
                        if (lane == 0 && !put_wsum(prev_slot, prev_lh, wacc)) fail(a.status, abort_flag, 44);
                        wacc = 0.f;
                    }
                }
                if (j == 0) {
                    // ---- the CTA's first slot: its state from the staging buffer into TMEM, as S~
                    // (sig = 1) and as S_before, and sum S_before^2
                    if (!mbar_wait_or_abort(&mb_st, 0, budget, abort_flag)) fail(a.status, abort_flag, 14);
                    st_seen = 1;
#pragma unroll
                    for (int g4 = 0; g4 < 4; ++g4) {
                        uint32_t sv[16];
#pragma unroll
                        for (int e = 0; e < 4; ++e) {
                            const float4 x = *reinterpret_cast<const float4*>(sbuf + sb_idx(r, 16 * hh + 4 * g4 + e));
                            den = fmaf(x.x, x.x, den); den = fmaf(x.y, x.y, den);
                            den = fmaf(x.z, x.z, den); den = fmaf(x.w, x.w, den);
                            sv[4 * e] = __float_as_uint(x.x); sv[4 * e + 1] = __float_as_uint(x.y);
                            sv[4 * e + 2] = __float_as_uint(x.z); sv[4 * e + 3] = __float_as_uint(x.w);
                        }
                        tmem_st16(tm + lane_off + TM_S + 64 * hh + 16 * g4, sv);
                        tmem_st16(tm + lane_off + TM_SB + 64 * hh + 16 * g4, sv);
                    }
                    warp_arrive(&mb_sfree, lane);                    // the staging buffer has been read
                    if (!make_k32(0)) fail(a.status, abort_flag, 16);
                    tmem_st_wait();
                    tc_fence_before();
                    warp_arrive(&mb_sready, lane);
                }
                // ---- E(j) is complete (and MMA_X(j) has read the state and K in fp32)
                if (!mbar_wait_or_abort(&mb_u, j & 1, budget, abort_flag)) fail(a.status, abort_flag, 10);
                if (!mbar_wait_or_abort(&mb_ifull[j & 3], (j >> 2) & 1, budget, abort_flag)) fail(a.status, abort_flag, 11);
                tc_fence_after();
                const float* cs = cst + (j & 3) * kConstWords;
                const float pass_f = cs[33];
                const float sig_after = cs[32];
                float wf[16];
#pragma unroll
                for (int e = 0; e < 4; ++e) {
                    const float4 w4 = *reinterpret_cast<const float4*>(cs + 16 * hh + 4 * e);
                    wf[4 * e] = w4.x; wf[4 * e + 1] = w4.y; wf[4 * e + 2] = w4.z; wf[4 * e + 3] = w4.w;
                }
                if (pass_f >= 0.f) {
                    // the decay would take the deferred scale out of range: S~ <- p S~ (MMA_S(j) has not
                    // been issued: it waits for this pass)
#pragma unroll
                    for (int g2 = 0; g2 < 2; ++g2) {
                        float sv[32];
                        tmem_ld32(tm + lane_off + TM_S + 64 * hh + 32 * g2, sv);
                        tmem_ld_wait();
#pragma unroll
                        for (int e = 0; e < 32; ++e) sv[e] *= pass_f;
                        tmem_st32(tm + lane_off + TM_S + 64 * hh + 32 * g2, sv);
                    }
                }
                {   // ---- pass: E = hi-half product + lo-half product (+ the X term), over this
                    // thread's 16 token columns, split into the packed (hi, lo) A operand of MMA_S
                    const uint32_t eb = tm + lane_off + TM_E + (j & 1) * 64 + 16 * hh;
                    float e0[16], e1[16];
                    tmem_ld16(eb, e0);
                    tmem_ld16(eb + 32, e1);
                    tmem_ld_wait();
#pragma unroll
                    for (int i = 0; i < 16; ++i) e0[i] += e1[i];
                    if (want_w) {
                        // squares summed over the warp's 32 rows, column by column: halving exchanges
                        // leave lanes 2c and 2c + 1 with column c of the 16
                        float x[16];
#pragma unroll
                        for (int i = 0; i < 16; ++i) x[i] = e0[i] * e0[i];
#pragma unroll
                        for (int w = 8, bit = 16; w >= 1; w >>= 1, bit >>= 1) {
                            const bool up = (lane & bit) != 0;
#pragma unroll
                            for (int i = 0; i < w; ++i) {
                                const float send = up ? x[i] : x[i + w];
                                x[i] = (up ? x[i + w] : x[i]) + __shfl_xor_sync(0xffffffffu, send, bit);
                            }
                        }
                        x[0] += __shfl_xor_sync(0xffffffffu, x[0], 1);
                        const int c = lane >> 1;
                        float f = wf[0];
#pragma unroll
                        for (int i = 1; i < 16; ++i) f = (c == i) ? wf[i] : f;
                        if ((lane & 1) == 0) atomicAdd(&s_u2[j & 1][16 * hh + c], x[0] * f * f);
                    }
                    uint32_t hi[8], lo[8];
#pragma unroll
                    for (int i = 0; i < 8; ++i) split2(e0[2 * i], e0[2 * i + 1], hi[i], lo[i]);
                    tmem_st8(tm + lane_off + TM_AP + 8 * hh, hi);
                    tmem_st8(tm + lane_off + TM_AP + 16 + 8 * hh, lo);
                    tmem_st_wait();
                }
                tc_fence_before();
                warp_arrive(&mb_uready, lane);
                warp_arrive(&mb_iempty[j & 3], lane);            // images and constants read
                sig = sig_after;
                // ---- while MMA_S(j) runs: the next sub-tile's K in fp32
                if (j + 1 < NS && !make_k32(j + 1)) fail(a.status, abort_flag, 16);
                if (!last) {
                    if (j + 1 < NS) warp_arrive(&mb_sready, lane);
                } else {
                    // ---- slot boundary: S_after = sig S~ out through the staging buffer, the next
                    // slot's state (staged meanwhile) into TMEM, drift partials against S_before
                    const bool has_next = j + 1 < NS;             // uniform
                    // a last slot that ends a head begun by CTA i - 1: S_before is not in TMEM (the
                    // slot started from the handed-over state) but staged, and its square sum is
                    // taken here
                    const bool shared_end = sch.is_suffix(slot);
                    float den_end = 0.f;
                    bool ok = mbar_wait_or_abort(&mb_s, j & 1, budget, abort_flag);
                    if (!ok) fail(a.status, abort_flag, 12);
                    if (!mbar_wait_or_abort(&mb_st, st_seen & 1, budget, abort_flag)) {
                        fail(a.status, abort_flag, 14);
                        ok = false;
                    }
                    ++st_seen;
                    tc_fence_after();
                    float num = 0.f, den_next = 0.f;
                    if (ok) {
#pragma unroll 1
                        for (int g4 = 0; g4 < 4; ++g4) {
                            const uint32_t col = 64 * hh + 16 * g4;
                            const int ch = 16 * hh + 4 * g4;      // this group's 16-byte chunks of row r
                            float sa[16], sb[16];
                            tmem_ld16(tm + lane_off + TM_S + col, sa);
                            if (shared_end) {
#pragma unroll
                                for (int e = 0; e < 4; ++e) {
                                    const float4 x = *reinterpret_cast<const float4*>(sbuf + sb_idx(r, ch + e));
                                    sb[4 * e] = x.x; sb[4 * e + 1] = x.y; sb[4 * e + 2] = x.z; sb[4 * e + 3] = x.w;
                                }
#pragma unroll
                                for (int e = 0; e < 16; ++e) den_end = fmaf(sb[e], sb[e], den_end);
                            } else {
                                tmem_ld16(tm + lane_off + TM_SB + col, sb);
                            }
                            tmem_ld_wait();
#pragma unroll
                            for (int e = 0; e < 16; ++e) {
                                sa[e] *= sig;
                                const float d = sa[e] - sb[e];
                                num = fmaf(d, d, num);
                            }
                            if (has_next) {
                                uint32_t sn[16];
#pragma unroll
                                for (int e = 0; e < 4; ++e) {
                                    const float4 x = *reinterpret_cast<const float4*>(sbuf + sb_idx(r, ch + e));
                                    den_next = fmaf(x.x, x.x, den_next); den_next = fmaf(x.y, x.y, den_next);
                                    den_next = fmaf(x.z, x.z, den_next); den_next = fmaf(x.w, x.w, den_next);
                                    sn[4 * e] = __float_as_uint(x.x); sn[4 * e + 1] = __float_as_uint(x.y);
                                    sn[4 * e + 2] = __float_as_uint(x.z); sn[4 * e + 3] = __float_as_uint(x.w);
                                }
                                tmem_st16(tm + lane_off + TM_S + col, sn);
                                tmem_st16(tm + lane_off + TM_SB + col, sn);
                            }
#pragma unroll
                            for (int e = 0; e < 4; ++e)
                                *reinterpret_cast<float4*>(sbuf + sb_idx(r, ch + e)) =
                                    make_float4(sa[4 * e], sa[4 * e + 1], sa[4 * e + 2], sa[4 * e + 3]);
                        }
                        tmem_st_wait();
                    }
                    tc_fence_before();
                    fence_async_smem();                          // S_after -> the state warp's TMA store
                    warp_arrive(&mb_sfree, lane);
                    if (has_next) warp_arrive(&mb_sready, lane);  // the next slot's state is in TMEM
                    // partial sums: pairwise in fp32, over the warp's lanes and then over the warps
                    float fn = num, fd = shared_end ? den_end : den;
#pragma unroll
                    for (int m = 16; m >= 1; m >>= 1) {
                        fn += __shfl_xor_sync(0xffffffffu, fn, m);
                        fd += __shfl_xor_sync(0xffffffffu, fd, m);
                    }
                    if (lane == 0) { s_red[0][warp] = fn; s_red[1][warp] = fd; }
                    if (named_sync_or(kBarChain, kChain, !ok)) { stop = true; break; }
                    if (warp == 0 && a.partials != nullptr && !sch.is_prefix(slot)) {   // a shared head: at its end
                        float pn = lane < kChainWarps ? s_red[0][lane] : 0.f;
                        float pd = lane < kChainWarps ? s_red[1][lane] : 0.f;
#pragma unroll
                        for (int m = kChainWarps / 2; m >= 1; m >>= 1) {
                            pn += __shfl_xor_sync(0xffffffffu, pn, m);
                            pd += __shfl_xor_sync(0xffffffffu, pd, m);
                        }
                        if (lane == 0) {
                            a.partials[(size_t)lh * 2 + 0] = pn;
                            a.partials[(size_t)lh * 2 + 1] = pd;
                        }
                    }
                    den = den_next;
                    sig = 1.f;
                }
                prev_lh = lh;
                prev_slot = slot;
                prev_last = last;
            }
            cc.next(sch, a);
        }
        // the CTA's last sub-tile (always a slot's last) once every warp's pass has added to it
        if (want_w && NS > 0 && !named_sync_or(kBarChain, kChain, *abort_flag) && warp == 0) {
            fold_writes(NS - 1);
            if (lane == 0 && !put_wsum(prev_slot, prev_lh, wacc)) fail(a.status, abort_flag, 45);
        }
    }

    tc_fence_before();
    __syncthreads();
    if (warp == kMmaWarp) {
        tc_fence_after();
        tmem_dealloc(tm, kTmemCols);
    }
}

typedef CUresult (*EncodeTiledFn)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*, const cuuint64_t*,
                                  const cuuint64_t*, const cuuint32_t*, const cuuint32_t*, CUtensorMapInterleave,
                                  CUtensorMapSwizzle, CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

EncodeTiledFn encode_fn() {
    static EncodeTiledFn fn = []() -> EncodeTiledFn {
        cudaDriverEntryPointQueryResult q;
        void* p = nullptr;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) == cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            return reinterpret_cast<EncodeTiledFn>(p);
        return nullptr;
    }();
    return fn;
}

// [L][T][H][128] bfloat16 as a 4-D map (d, H, T, L): a box of 64 features x 1 head x `rows` tokens,
// 128-byte swizzle; tokens past T read as zero.
bool make_map(CUtensorMap* map, const void* base, int L, int T, int H, int rows) {
    EncodeTiledFn enc = encode_fn();
    if (!enc) return false;
    cuuint64_t dims[4] = {(cuuint64_t)kD, (cuuint64_t)H, (cuuint64_t)T, (cuuint64_t)L};
    cuuint64_t strides[3] = {(cuuint64_t)kD * 2, (cuuint64_t)H * kD * 2, (cuuint64_t)T * H * kD * 2};
    cuuint32_t box[4] = {64, 1, (cuuint32_t)rows, 1};
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

// Scratch (past the workspace header): the hand-over area for up to one CTA per SM: states
// [grid][128][128] fp32, write-size sums [grid].
struct TcScratch {
    size_t ho_state, ho_wsum, total;
};

TcScratch tc_scratch_layout(int L, int Hv) {
    const int grid = std::max(1, std::min(L * Hv, device_sm_count()));
    TcScratch l;
    l.ho_state = 0;
    l.ho_wsum = (size_t)grid * kD * kD * 4;
    l.total = l.ho_wsum + (size_t)grid * 4;
    return l;
}

// Equal tile runs, with heads split between neighbouring CTAs, when they shorten the slowest CTA:
// a slot boundary costs about `kBoundary` tiles and a hand-over about `kHandOver`.
constexpr double kBoundary = 0.6, kHandOver = 2.0;

}  // namespace

size_t gdn_tc_scratch_bytes(int L, int Hv, int dk, int dv, int dtype, int T) {
    if (dk != kD || dv != kD || dtype != DELTAS_BF16 || L <= 0 || Hv <= 0 || T <= 0) return 0;
    return tc_scratch_layout(L, Hv).total;
}

bool gdn_tc_shape(const GdnArgs& a) {
    return a.dk == kD && a.dv == kD && a.dtype == DELTAS_BF16 && a.out == nullptr && a.T > 0;
}

bool gdn_tc_supported(const GdnArgs& a) {
    return gdn_tc_shape(a) &&
           (long long)a.L * a.Hv * kD < (1ll << 31) &&                          // TMA row coordinate
           a.Hk <= (1 << 24) && a.T < (1 << 30) &&
           a.scratch != nullptr &&
           a.scratch_bytes >= gdn_tc_scratch_bytes(a.L, a.Hv, a.dk, a.dv, a.dtype, a.T) &&
           std::min(a.L * a.Hv, device_sm_count()) <= 512 &&                    // hand-over bits
           encode_fn() != nullptr;
}

cudaError_t launch_gdn_update_tc(const GdnArgs& a, cudaStream_t s) {
    const TcScratch sl = tc_scratch_layout(a.L, a.Hv);
    const int sms = device_sm_count();
    const int H = a.L * a.Hv;
    const int grid = std::min(H, sms);
    CUtensorMap kmap, vmap, smap, hmap;
    if (!make_map(&kmap, a.k, a.L, a.T, a.Hk, kTile) || !make_map(&vmap, a.v, a.L, a.T, a.Hv, kC) ||
        !make_state_map(&smap, a.state, H) || !make_state_map(&hmap, a.scratch + sl.ho_state, grid))
        return cudaErrorInvalidValue;
    // The attribute is per device; setting it on every launch costs little and stays correct after
    // a device reset and from any host thread.
    cudaError_t e = cudaFuncSetAttribute(gdn_fused_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         (int)kSmemAlloc);
    if (e != cudaSuccess) return e;
    const int n_tiles = (a.T + kTile - 1) / kTile;
    TcArgs t;
    t.L = a.L; t.Hk = a.Hk; t.Hv = a.Hv; t.T = a.T; t.n_tiles = n_tiles;
    t.g = a.g; t.beta = a.beta;
    t.state = a.state; t.partials = a.partials; t.wnorm = a.wnorm; t.status = a.status;
    t.ho_bits = reinterpret_cast<uint32_t*>(a.status) + 4;
    t.ho_wsum = reinterpret_cast<float*>(a.scratch + sl.ho_wsum);
    t.split = 0;
    if (H > grid && H % grid != 0) {
        const double whole = std::ceil((double)H / grid) * (n_tiles + kBoundary);
        const double runs = std::ceil((double)H * n_tiles / grid);
        const double parted = runs + (runs / n_tiles + 2.0) * kBoundary + kHandOver;
        t.split = parted < whole ? 1 : 0;
    }
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(grid);
    cfg.blockDim = dim3(kThreads);
    cfg.dynamicSmemBytes = kSmemAlloc;
    cfg.stream = s;
    cudaLaunchAttribute attr[1];
    if (t.split) {
        // every CTA must be resident: a split head's second part waits for its first
        attr[0].id = cudaLaunchAttributeCooperative;
        attr[0].val.cooperative = 1;
        cfg.attrs = attr;
        cfg.numAttrs = 1;
        e = cudaLaunchKernelEx(&cfg, gdn_fused_kernel, kmap, vmap, smap, hmap, t);
        if (e != cudaErrorCooperativeLaunchTooLarge) return e;
        (void)cudaGetLastError();                 // fewer SMs than the grid: whole heads instead
        t.split = 0;
    }
    cfg.attrs = nullptr;
    cfg.numAttrs = 0;
    return cudaLaunchKernelEx(&cfg, gdn_fused_kernel, kmap, vmap, smap, hmap, t);
}

}  // namespace deltas
