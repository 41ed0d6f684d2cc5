// Gated delta rule over one chunk on the Blackwell tensor cores (tcgen05 + TMEM + TMA), d = 128,
// bfloat16 k/v, fp32 state, with the state-drift partials fused in: one persistent kernel.
//
// Paper: Sec. 3.2, Eq. 1/2 (the recurrence) and Eq. 3 (drift numerator / denominator per layer
// and head).  The chunk is processed in tiles of C = 64 tokens with the chunkwise (WY) form of
// Eq. 1.  Inside a tile let G be the inclusive cumulative log-decay, gamma_t = exp(G_t),
// gamma_C = exp(G_{C-1}), delta_t = gamma_C / gamma_t <= 1, and X = K S0^T (row t: S0 k_t).  With
//   A[t][i] = beta_t (gamma_t / gamma_i) k_t.k_i  (i < t),   U = (I + A)^-1 diag(beta) (V - diag(gamma) X)
// the state after the tile is S_C = gamma_C S0 + sum_t delta_t u_t k_t^T.  The decay factors out of
// the triangular solve by a diagonal similarity, I + A = diag(gamma) (I + diag(beta) L) diag(gamma)^-1
// with L the strictly lower part of K K^T, so with the decay-free
//   N_beta = (I + diag(beta) L)^-1 diag(beta)
// the decayed writes are  U~ = diag(delta) U = N_beta (diag(delta) V - gamma_C X):  every decay
// factor the kernel uses is at most 1, and the inverse depends on k and beta only.  The X term
// folds into one product with the state:  gamma_C X^T N_beta^T = S0 (K^T N_beta^T).
//
// Work split inside one CTA (one per SM, persistent over (layer, value head) slots):
//   producer (two groups of 4 warps, each taking every other tile, so that a group has two tile
//            periods for one tile): K K^T of the tile comes from the tensor core; the group forms
//            diag(beta) L, inverts I + diag(beta) L (16 x 16 diagonal blocks by substitution, then
//            two levels of block products) and writes two operand images, each a bfloat16
//            (hi, lo) pair laid out as the two K-halves of one operand:
//              B1 = u N_beta diag(delta)   and   B3 = N_beta
//            (u: the state's deferred scale, below)
//   MMA      (1 warp, one elected lane): every tcgen05.mma, each group's completion by commit
//   chain    (4 warps): the pass over E, the K^T N_beta^T product into the B operand W, head
//            boundaries (state in and out, drift partials)
//   loads    (1 warp): K and V tiles by TMA, L2 prefetch of the tiles ahead and of the next state
// Per tile j, in tensor-pipe order:
//   E(j)  += S~ W(j)                  (tf32: A = the fp32 state straight from TMEM)
//   Q(j+1) = K^T B3, E(j+1) = V^T B1  (bf16 (hi, lo); the chain turns Q into W(j+1) = -c Q^T in
//                                      tf32 in shared memory)
//   K K^T (j+2)                       (bf16, for the producer)
//   pass   (chain) E -> bfloat16 (hi, lo), in place
//   S~     = 2^-s S~ + E K            (the input state scaled by the instruction's power-of-two
//                                      scale-input-d operand)
// The tensor core does not order an MMA that reads a TMEM region as its A operand after an earlier
// MMA that wrote it (measured), so E += S~ W waits for the previous state update's commit.
//
// Deferred decay.  TMEM holds S~ with the true state S = sig S~.  A tile with decay gamma_C takes
// p = gamma_C sig and a shift s in [0, 15] that brings p 2^s into [1/2, 1) when it can: then
// sig <- p 2^s, u = 1 / sig, c = 2^-s, and the state update scales S~ by 2^-s as it accumulates
// (exact).  When p < 2^-45 (no shift reaches 2^-30) the chain multiplies S~ by p in a pass instead,
// sig restarts at 1, u = 1 and c = p.  So sig stays in [2^-30, 1] and u below 2^30.  The producer
// writes each tile's constants (sig after the tile, the shift, the pass factor, c, the write-size
// scales) beside its images.
//
// Precision.  k, v exact in bfloat16; K K^T exact in fp32.  E += S~ W reads S~ as tf32 (10
// explicit mantissa bits, truncated) and W is rounded to tf32: errors confined to the delta
// correction.  B1, B3 and E take two-term bfloat16 splits (x = hi + lo, about 2^-16 relative); the
// inverse is formed in fp32.  A CPU model of exactly these roundings gives a state error against
// fp64 of 2.6e-4 at the slowest decay the tests use (4 chunks of 1024 tokens), 5e-6 at a typical
// one, and drift numerators within 1.1e-4.
//
// Synchronisation.  Roles hand work to each other through mbarriers only; every wait is bounded
// (about one second, or the workspace header's override); a wait that runs out records
// DELTAS_ERR_TIMEOUT, raises a CTA-wide abort flag so the other roles stop waiting, and the CTA
// drains its MMAs and copies before freeing TMEM.  Heads split between neighbouring CTAs (equal
// tile runs, see ChainSched) hand the state over through the workspace with a bit per CTA boundary
// in the workspace header, which its reader clears after use.
//
// TMEM (512 columns, 128 lanes): S~ [0,128), S_before [128,256), E0 [256,320), E1 [320,384)
// (E fp32, then its (hi, lo) A operand in place), K K^T [384,448) (lanes 0..63), Q [448,512).
#include <algorithm>
#include <cmath>

#include "internal.cuh"
#include "tc_ptx.cuh"

namespace deltas {
namespace {

using namespace tc;

constexpr int kC = 64;                 // tokens per tile
constexpr int kD = 128;                // head dim (d_k = d_v)
constexpr float kHardMin = 0x1p-45f;   // p below this: the state is rescaled by a pass

// ---- roles
constexpr int kChainWarps = 4;         // warps 0..3: warp q serves TMEM lanes 32 q ..
constexpr int kChain = 32 * kChainWarps;
constexpr int kProdWarp0 = 4;          // warps 4..7: producer group 1 (odd tiles), 8..11: group 0 (even);
                                       // warp i of a group (i = warp % 4) reads TMEM lanes 32 i ..
constexpr int kProd = 128;             // threads of a producer group
constexpr int kMmaWarp = 12;
constexpr int kLoadWarp = 13;
constexpr int kThreads = 14 * 32;
constexpr int kBarChain = 1;           // named barriers: chain, producer group 0, group 1 (128 threads each)
constexpr int kBarProd = 2;

// ---- TMEM columns
constexpr uint32_t kTmemCols = 512;
constexpr uint32_t TM_S = 0, TM_SB = 128, TM_E = 256, TM_KK = 384, TM_Q = 448;

// ---- shared memory (bytes from a 1024-aligned base)
constexpr int kKSlots = 5;             // K ring: a tile's K K^T is issued three tiles before its state update
constexpr uint32_t SM_K = 0;           // 5 tiles x 16 KB: 2 column blocks (d 0-63, 64-127) x 64 rows x 128 B, SW128
constexpr uint32_t SM_V = 81920;       // 16 KB, same layout (also the K K^T product's over-read past the last
                                       // K tile: rows 64..127 of its M = 128 A)
constexpr uint32_t SM_B1 = 98304;      // 16 KB: rows t of u N_beta diag(delta): hi in column block 0, lo in
                                       // block 1 (64 rows x 128 B each, SW128)
constexpr uint32_t SM_B3 = 114688;     // 16 KB: N_beta, same layout
constexpr uint32_t SM_W = 131072;      // 32 KB: W^T = -c N_beta K in tf32, rows t: 4 column blocks (32 dims)
                                       // x 64 rows x 128 B, SW128 (the B operand of E += S~ W)
constexpr uint32_t SM_PW = 163840;     // producer workspaces, one per group
// A group's workspace (fp32): rows 0..31 of M = diag(beta) L and of N = (I + diag(beta) L)^-1 hold
// columns 0..31 only (the rest is above the diagonal), rows 32..63 all 64 columns; the block
// products; beta, delta and (u, c) of the group's tile, double-buffered (the constants warp writes
// the group's next tile's while the others may still read this one's).
constexpr int kTS = 36, kBS = 68, kPS = 36;   // row strides (16-byte aligned rows)
constexpr int PW_MT = 0, PW_MB = PW_MT + 32 * kTS, PW_NT = PW_MB + 32 * kBS, PW_NB = PW_NT + 32 * kTS,
              PW_P = PW_NB + 32 * kBS, PW_BETA = PW_P + 32 * kPS, PW_DELTA = PW_BETA + 128, PW_UC = PW_DELTA + 128,
              PW_FLOATS = PW_UC + 8;
constexpr uint32_t kPwBytes = PW_FLOATS * 4;
constexpr uint32_t SM_CONST = SM_PW + 2 * kPwBytes;   // 2 slots x kConstWords: per-tile constants
constexpr int kConstWords = 72;        // [0,64) write-size scale per token, 64 sig after, 65 pass factor
                                       // (< 0: none), 66 shift (int), 67 c
constexpr uint32_t SM_BYTES = SM_CONST + 2 * kConstWords * 4;
constexpr uint32_t kSmemAlloc = SM_BYTES + 1024;
static_assert(SM_V % 1024 == 0 && SM_B1 % 1024 == 0 && SM_B3 % 1024 == 0 && SM_W % 1024 == 0 &&
              kPwBytes % 16 == 0 && SM_CONST % 16 == 0, "shared-memory map");
static_assert(SM_V == SM_K + kKSlots * 16384 && SM_B1 == SM_V + 16384 && SM_B3 == SM_B1 + 16384 &&
              SM_W == SM_B3 + 16384 && SM_PW == SM_W + 32768, "map order");
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

// D (16 x 8) += A (16 x 16, row-major) B (16 x 8) on the warp's tensor-core path, bf16 in, fp32
// accumulate.  Fragments (g = lane / 4, t = lane % 4), each register a bf16 pair, lower k in the
// low half: a = A[g][2t..], A[g+8][2t..], A[g][2t+8..], A[g+8][2t+8..]; b = B[2t..][g],
// B[2t+8..][g]; d = D[g][2t, 2t+1], D[g+8][2t, 2t+1].
__device__ __forceinline__ void mma_m16n8k16_bf16(float (&d)[4], const uint32_t (&a)[4], const uint32_t (&b)[2]) {
    asm volatile("mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, "
                 "{%0,%1,%2,%3};"
                 : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
                 : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b[0]), "r"(b[1]));
}

// D (16 x 8) += A (16 x 16 KS) B (16 KS x 8) for fp32 operands in shared memory (A row-major with
// row stride lda, B row-major B[k][n] with row stride ldb), each split into bfloat16 (hi, lo) in
// registers and multiplied as lo hi + hi lo + hi hi (about 2^-16 relative error per product).
template <int KS>
__device__ __forceinline__ void mma_f32_split(float (&d)[4], const float* A, int lda, const float* B, int ldb,
                                              int g, int t) {
    // the three products accumulate separately (independent chains), summed at the end
    float d1[4] = {0.f, 0.f, 0.f, 0.f}, d2[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
    for (int ks = 0; ks < KS; ++ks) {
        const float* a0 = A + g * lda + 16 * ks + 2 * t;
        const float2 x0 = *reinterpret_cast<const float2*>(a0);
        const float2 x1 = *reinterpret_cast<const float2*>(a0 + 8 * lda);
        const float2 x2 = *reinterpret_cast<const float2*>(a0 + 8);
        const float2 x3 = *reinterpret_cast<const float2*>(a0 + 8 * lda + 8);
        const float* b0 = B + (16 * ks + 2 * t) * ldb + g;
        uint32_t ah[4], al[4], bh[2], bl[2];
        split2(x0.x, x0.y, ah[0], al[0]);
        split2(x1.x, x1.y, ah[1], al[1]);
        split2(x2.x, x2.y, ah[2], al[2]);
        split2(x3.x, x3.y, ah[3], al[3]);
        split2(b0[0], b0[ldb], bh[0], bl[0]);
        split2(b0[8 * ldb], b0[9 * ldb], bh[1], bl[1]);
        mma_m16n8k16_bf16(d1, al, bh);
        mma_m16n8k16_bf16(d2, ah, bl);
        mma_m16n8k16_bf16(d, ah, bh);
    }
#pragma unroll
    for (int i = 0; i < 4; ++i) d[i] += d1[i] + d2[i];
}

// One kind::f16 MMA from TMEM A that scales the accumulator it reads by 2^-shift (the
// instruction's scale-input-d operand, an immediate: D = A B + 2^-shift D), shift in [0, 15].
template <int S>
__device__ __forceinline__ void mma_bf16_ta_scaled(uint32_t d, uint32_t a, uint64_t b, uint32_t idesc) {
    asm volatile("{\n\t.reg .pred q;\n\t"
                 "setp.eq.b32 q, %3, %3;\n\t"
                 "tcgen05.mma.cta_group::1.kind::f16 [%0], [%1], %2, %3, q, %4;\n\t}"
                 :: "r"(d), "r"(a), "l"(b), "r"(idesc), "n"(S) : "memory");
}
__device__ __noinline__ void mma_bf16_ta_shift_1t(int shift, uint32_t d, uint32_t a, uint64_t b, uint32_t idesc) {
    switch (shift) {
        case 0: mma_bf16_ta_scaled<0>(d, a, b, idesc); break;
        case 1: mma_bf16_ta_scaled<1>(d, a, b, idesc); break;
        case 2: mma_bf16_ta_scaled<2>(d, a, b, idesc); break;
        case 3: mma_bf16_ta_scaled<3>(d, a, b, idesc); break;
        case 4: mma_bf16_ta_scaled<4>(d, a, b, idesc); break;
        case 5: mma_bf16_ta_scaled<5>(d, a, b, idesc); break;
        case 6: mma_bf16_ta_scaled<6>(d, a, b, idesc); break;
        case 7: mma_bf16_ta_scaled<7>(d, a, b, idesc); break;
        case 8: mma_bf16_ta_scaled<8>(d, a, b, idesc); break;
        case 9: mma_bf16_ta_scaled<9>(d, a, b, idesc); break;
        case 10: mma_bf16_ta_scaled<10>(d, a, b, idesc); break;
        case 11: mma_bf16_ta_scaled<11>(d, a, b, idesc); break;
        case 12: mma_bf16_ta_scaled<12>(d, a, b, idesc); break;
        case 13: mma_bf16_ta_scaled<13>(d, a, b, idesc); break;
        case 14: mma_bf16_ta_scaled<14>(d, a, b, idesc); break;
        default: mma_bf16_ta_scaled<15>(d, a, b, idesc); break;
    }
}

// The waits of this kernel: one try inline, the bounded loop out of line (the kernel's code must
// stay small: every role's loop shares the SM's instruction cache, and misses are served from a
// busy L2).
__device__ __noinline__ bool wait_slow(uint64_t* bar, uint32_t parity, uint64_t budget_ns,
                                       const volatile int* abort) {
    const long long t0 = clock64();
    const long long budget = (long long)(budget_ns * 2);
    for (;;) {
        if (mbar_try_wait_sleep(bar, parity, 20000u)) return true;
        if (*abort) return false;
        if (clock64() - t0 > budget) return false;
    }
}
__device__ __forceinline__ bool wait_bar(uint64_t* bar, uint32_t parity, uint64_t budget_ns,
                                         const volatile int* abort) {
    if (mbar_try_wait(bar, parity)) return true;
    return wait_slow(bar, parity, budget_ns, abort);
}

// All lanes of a converged warp wait; the result is the same on every lane.
__device__ __forceinline__ bool warp_wait(uint64_t* bar, uint32_t parity, uint64_t budget_ns,
                                          const volatile int* abort) {
    const bool ok = wait_bar(bar, parity, budget_ns, abort);
    return __all_sync(0xffffffffu, ok) != 0;
}

__device__ __noinline__ void fail(int32_t* status, volatile int* abort, int where) {
    record_status(status, DELTAS_ERR_TIMEOUT, where);
    *abort = 1;
}

// One arrival per warp: every lane's TMEM stores / shared-memory writes were completed and fenced
// before the __syncwarp; lane 0 then arrives (release).
__device__ __forceinline__ void warp_arrive(uint64_t* bar, int lane) {
    __syncwarp();
    if (lane == 0) mbar_arrive(bar);
}

__device__ __forceinline__ uint32_t ld_acquire(const uint32_t* p) {
    uint32_t v;
    asm volatile("ld.acquire.gpu.global.b32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
    return v;
}

__device__ __forceinline__ void prefetch_l2(const void* p) {
    asm volatile("prefetch.global.L2 [%0];" :: "l"(p) : "memory");
}

__device__ __forceinline__ void prefetch_l2_bulk(const void* p, uint32_t bytes) {
    asm volatile("cp.async.bulk.prefetch.L2.global [%0], %1;" :: "l"(p), "r"(bytes) : "memory");
}

// The per-tile decay bookkeeping (see the header): from p = gamma_C sig, the shift s, the scale u
// of the V term, the coefficient c of the state term, the pass factor (< 0: no pass) and sig after
// the tile.
struct DecayStep {
    int shift;
    float u, c, pass, sig;
};
__device__ __forceinline__ DecayStep decay_step(float p) {
    DecayStep d;
    if (!(p >= kHardMin)) {
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
    float* state;                // [L * Hv][128][128]
    float* partials;
    float* wnorm;
    int32_t* status;
    uint32_t* ho_bits;           // hand-over bits in the workspace header: [0, 16) state, [16, 32) sums
    float* ho_state;             // [grid][128][128]
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
    __device__ __noinline__ void set_slot(int slot, const ChainSched& sc, const TcArgs& a) {
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

// 16 fp32 of a state row, global -> registers (through L2 only for data another CTA wrote)
__device__ __forceinline__ void ld16_global(const float* p, float (&v)[16], bool cache_global) {
#pragma unroll
    for (int e = 0; e < 4; ++e) {
        const float4 x = cache_global ? __ldcg(reinterpret_cast<const float4*>(p) + e)
                                      : __ldg(reinterpret_cast<const float4*>(p) + e);
        v[4 * e] = x.x; v[4 * e + 1] = x.y; v[4 * e + 2] = x.z; v[4 * e + 3] = x.w;
    }
}

__global__ void __launch_bounds__(kThreads, 1)
gdn_fused_kernel(const __grid_constant__ CUtensorMap kmap, const __grid_constant__ CUtensorMap vmap, TcArgs a)
{
    extern __shared__ uint8_t smem_raw[];
    uint8_t* sm = smem_raw + ((1024 - (smem_u32(smem_raw) & 1023)) & 1023);
    // loads -> roles: K, V tiles full; MMA -> loader: their empties.  producer -> MMA / chain: images
    // and constants full (ifull, by tile parity); the images are free once their products have
    // completed (bfree, by the parity of the tile that used them), the constants once the chain has
    // read them (iempty).  MMA -> producer group: K K^T done (kk, by parity); producer -> MMA: read
    // (kkfree).  MMA -> chain: Q done (q), E ready (u), state updated (s); chain -> MMA: W and the
    // slot's state ready (ready), E packed (uready).
    __shared__ uint64_t mb_kfull[kKSlots], mb_kempty[kKSlots], mb_vfull, mb_vempty, mb_ifull[2], mb_iempty[2];
    __shared__ uint64_t mb_bfree[2], mb_kk[2], mb_kkfree, mb_q, mb_ready, mb_u, mb_uready, mb_s, mb_fin;
    __shared__ uint32_t s_tmem;
    __shared__ int s_abort;
    __shared__ float s_red[2][kChainWarps];
    __shared__ float s_u2[2][kC];                     // per-token squared write sizes (tile parity)
    volatile int* abort_flag = &s_abort;

    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    // bounded-wait budget: the workspace header's override (microseconds) or about one second
    const uint32_t budget_us = reinterpret_cast<const volatile uint32_t*>(a.status)[2];
    const uint64_t budget = budget_us ? (uint64_t)budget_us * 1000ull : kWaitBudgetNs;
    ChainSched sch;
    sch.init(a);
    const int NJ = sch.NJ;                            // tiles of this CTA
    const int me = (int)blockIdx.x;
    uint32_t* bits_state = a.ho_bits;
    uint32_t* bits_wsum = a.ho_bits + 16;

    if (warp == kMmaWarp) {
        tmem_alloc(&s_tmem, kTmemCols);
        tmem_relinquish();
        if (lane == 0) {
            for (int b = 0; b < kKSlots; ++b) { mbar_init(&mb_kfull[b], 1); mbar_init(&mb_kempty[b], 1); }
            mbar_init(&mb_vfull, 1); mbar_init(&mb_vempty, 1);
            for (int b = 0; b < 2; ++b) {
                mbar_init(&mb_ifull[b], 4); mbar_init(&mb_iempty[b], kChainWarps);
                mbar_init(&mb_bfree[b], 1); mbar_init(&mb_kk[b], 1);
            }
            mbar_init(&mb_kkfree, 2); mbar_init(&mb_q, 1);
            mbar_init(&mb_ready, kChainWarps); mbar_init(&mb_u, 1); mbar_init(&mb_uready, kChainWarps);
            mbar_init(&mb_s, 1); mbar_init(&mb_fin, 1);
            fence_barrier_init();
        }
    }
    if (warp == kLoadWarp && lane == 0) { prefetch_tensormap(&kmap); prefetch_tensormap(&vmap); }
    if (tid == 0) s_abort = 0;
    if (tid < 2 * kC) s_u2[tid >> 6][tid & (kC - 1)] = 0.f;
    grid_dep_launch();                                // the next kernel (the score) may be scheduled
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tm = s_tmem;
    float* cst = reinterpret_cast<float*>(sm + SM_CONST);

    if (warp == kMmaWarp) {
        // =========================================================== MMA issue (converged warp;
        // one elected lane issues each group and commits it)
        const uint32_t idW = idesc_bf16(128, 64, 1, 0);   // Q and E products: A MN-major (K^T, V^T)
        const uint32_t idX = idesc_tf32(128, 64);
        const uint32_t idS = idesc_bf16(128, 128, 0, 1);
        const uint32_t idK = idesc_bf16(128, 64, 0, 0);
        // K K^T of tile J (M = 128: rows 64..127 of A read the 16 KB past the tile; their output
        // lanes are ignored), once the tile has landed and the producer has read the previous one
        // (every product below is a rolled loop of single MMAs from one elected lane: the issue
        // rate is the tensor pipe's, and the code stays small)
        auto issue_kk = [&](int J) -> bool {
            if (!warp_wait(&mb_kfull[J % kKSlots], (J / kKSlots) & 1, budget, abort_flag)) return false;
            if (J > 0 && !warp_wait(&mb_kkfree, (J - 1) & 1, budget, abort_flag)) return false;
            tc_fence_after();
            if (elect_one()) {
                const uint32_t base = smem_u32(sm + SM_K + (J % kKSlots) * 16384);
#pragma unroll 1
                for (int s = 0; s < 8; ++s) {
                    const uint64_t d = sdesc_sw128(base + (s >> 2) * 8192 + (s & 3) * 32, 16, 1024);
                    mma_bf16_1t(tm + TM_KK, d, d, idK, s > 0);
                }
            }
            __syncwarp();
            mma_commit(&mb_kk[J & 1]);
            return true;
        };
        // A (K^T or V^T: the tile read MN-major; k-steps 4..7 repeat tokens 0..63 for the lo half)
        // times B (an image: k-steps 0..3 its hi block, 4..7 its lo block) into D
        auto issue_img = [&](uint32_t d, uint32_t a_base, uint32_t b_base) {
            if (elect_one()) {
#pragma unroll 1
                for (int s = 0; s < 8; ++s)
                    mma_bf16_1t(d, sdesc_sw128(a_base + (s & 3) * 2048, 8192, 1024),
                                sdesc_sw128(b_base + (s >> 2) * 8192 + (s & 3) * 32, 16, 1024), idW, s > 0);
            }
            __syncwarp();
        };
        // Q(J) = K(J)^T B3(J) and E(J) = V(J)^T B1(J), once the images are written
        auto issue_images = [&](int J) -> bool {
            if (!warp_wait(&mb_ifull[J & 1], (J >> 1) & 1, budget, abort_flag)) return false;
            tc_fence_after();
            issue_img(tm + TM_Q, smem_u32(sm + SM_K + (J % kKSlots) * 16384), smem_u32(sm + SM_B3));
            mma_commit(&mb_q);
            if (!warp_wait(&mb_vfull, J & 1, budget, abort_flag)) return false;
            tc_fence_after();
            issue_img(tm + TM_E + (J & 1) * 64, smem_u32(sm + SM_V), smem_u32(sm + SM_B1));
            mma_commit(&mb_vempty);
            mma_commit(&mb_bfree[J & 1]);              // the images' last reader
            return true;
        };
        bool ok = true;
        if (NJ > 0) {
            for (int J = 0; ok && J < 3 && J < NJ; ++J) ok = issue_kk(J);
            if (ok) ok = issue_images(0);
            if (!ok) fail(a.status, abort_flag, 1);
        }
        for (int j = 0; ok && j < NJ; ++j) {
            const uint32_t eb = tm + TM_E + (j & 1) * 64;
            int shift = 0;
            {   // E(j) += S~ W(j) (A: the state from TMEM as tf32, 8 columns per K = 8 step; B: W in
                // tf32).  E(j)'s own product was issued before, into the same accumulator.
                if (!warp_wait(&mb_ready, j & 1, budget, abort_flag)) { fail(a.status, abort_flag, 2); break; }
                if (j > 0 && !warp_wait(&mb_s, (j - 1) & 1, budget, abort_flag)) { fail(a.status, abort_flag, 3); break; }
                // E(j)'s own product has completed: for j > 0 the state update's commit covers it
                // (issued after it), for the first tile its own commit
                if (j == 0 && !warp_wait(&mb_vempty, 0, budget, abort_flag)) { fail(a.status, abort_flag, 7); break; }
                // the tile's images and constants are held until the chain has read them
                shift = reinterpret_cast<const volatile int*>(cst + (j & 1) * kConstWords)[66];
                tc_fence_after();
                if (elect_one()) {
                    const uint32_t wb = smem_u32(sm + SM_W);
#pragma unroll 1
                    for (int s = 0; s < 16; ++s)
                        mma_tf32_ta_1t(eb, tm + TM_S + 8 * s, sdesc_sw128(wb + (s >> 2) * 8192 + (s & 3) * 32, 16, 1024),
                                       idX, 1);
                }
                __syncwarp();
                mma_commit(&mb_u);
            }
            // K K^T three tiles ahead (a producer group has two tile periods for its tile), the next
            // tile's Q and E, while the chain runs its pass
            if (j + 3 < NJ && !issue_kk(j + 3)) { fail(a.status, abort_flag, 5); break; }
            if (j + 1 < NJ && !issue_images(j + 1)) { fail(a.status, abort_flag, 4); break; }
            {   // S~ = 2^-shift S~ + E K  (A: E hi / lo packed in place; K read MN-major)
                if (!warp_wait(&mb_uready, j & 1, budget, abort_flag)) { fail(a.status, abort_flag, 6); break; }
                tc_fence_after();
                if (elect_one()) {
                    // K-step s: A = E's hi (s < 4) or lo (s >= 4) columns of token block s & 3
                    const uint32_t kb = smem_u32(sm + SM_K + (j % kKSlots) * 16384);
                    mma_bf16_ta_shift_1t(shift, tm + TM_S, eb, sdesc_sw128(kb, 8192, 1024), idS);
#pragma unroll 1
                    for (int s = 1; s < 8; ++s) {
                        const int tb = s & 3;
                        mma_bf16_ta_1t(tm + TM_S, eb + 32 * (tb >> 1) + 8 * (tb & 1) + 16 * (s >> 2),
                                       sdesc_sw128(kb + tb * 2048, 8192, 1024), idS, 1);
                    }
                }
                __syncwarp();
                mma_commit(&mb_s);
                mma_commit(&mb_kempty[j % kKSlots]);   // the tile's last reader
            }
        }
        if (__any_sync(0xffffffffu, *abort_flag != 0)) {
            mma_commit(&mb_fin);                       // every MMA this warp issued has completed
            mbar_wait(&mb_fin, 0, budget);
        }
        __syncwarp();
    } else if (warp == kLoadWarp) {
        // =========================================================== K and V tiles, each into its
        // buffer once the MMA that last read the buffer has completed.  The V stream runs two tiles
        // behind the K stream: the MMA takes K three tiles ahead of the state update (for K K^T) but
        // V one tile ahead, so a V load held for its buffer must not hold up the K loads behind it.
        // The tiles ahead of the K ring and each slot's successor's state are prefetched into L2.
        TileCursor kc, vc, pf;
        kc.init(sch, a);
        vc = kc;
        pf = kc;
        int kp[kKSlots], vp = -1;                      // last tile loaded per buffer
        for (int b = 0; b < kKSlots; ++b) kp[b] = -1;
        grid_dep_wait();
        auto prefetch_tile = [&](const TileCursor& c) {    // all lanes
            if (lane == 0) {
                tma_prefetch_4d(&kmap, 0, c.kh, c.jt * kC, c.l);
                tma_prefetch_4d(&kmap, 64, c.kh, c.jt * kC, c.l);
                tma_prefetch_4d(&vmap, 0, c.h, c.jt * kC, c.l);
                tma_prefetch_4d(&vmap, 64, c.h, c.jt * kC, c.l);
            }
            // the tile's g and beta (one 4-byte value per token, a line apart): the producer reads
            // them one group-tile ahead, too late to take an HBM miss off its path
            const int t0 = c.jt * kC + lane;
            const size_t i0 = ((size_t)c.l * a.T + t0) * a.Hv + c.h;
            if (t0 < a.T) { prefetch_l2(a.g + i0); prefetch_l2(a.beta + i0); }
            if (t0 + 32 < a.T) { prefetch_l2(a.g + i0 + 32 * (size_t)a.Hv); prefetch_l2(a.beta + i0 + 32 * (size_t)a.Hv); }
        };
        for (int i = 0; i < kKSlots && i < NJ; ++i) {
            prefetch_tile(pf);
            __syncwarp();
            pf.next(sch, a);
        }
        constexpr int kVLag = 2;
        bool ok = true;
        for (int n = 0; ok && n < NJ + kVLag; ++n) {
            if (n < NJ) {                                // K of tile n
                if (n + kKSlots < NJ) {
                    prefetch_tile(pf);
                    __syncwarp();
                    pf.next(sch, a);
                }
                if (kc.jt == kc.tb && kc.k + 1 < sch.n_slots && !sch.is_suffix(kc.k + 1) && elect_one()) {
                    int lh, tb, te;                      // the next slot's state, ahead of its boundary
                    sch.slot(kc.k + 1, a.n_tiles, lh, tb, te);
                    prefetch_l2_bulk(a.state + (size_t)lh * kD * kD, kD * kD * 4);
                }
                __syncwarp();
                const int bk = n % kKSlots;
                if (n >= kKSlots && !warp_wait(&mb_kempty[bk], ((n / kKSlots) - 1) & 1, budget, abort_flag)) {
                    fail(a.status, abort_flag, 30); break;
                }
                if (elect_one()) {
                    uint8_t* dst = sm + SM_K + bk * 16384;
                    mbar_arrive_expect_tx(&mb_kfull[bk], 16384);
                    tma_load_4d(dst, &kmap, &mb_kfull[bk], 0, kc.kh, kc.jt * kC, kc.l);
                    tma_load_4d(dst + 8192, &kmap, &mb_kfull[bk], 64, kc.kh, kc.jt * kC, kc.l);
                }
                __syncwarp();
                kp[bk] = n;
                kc.next(sch, a);
            }
            const int m = n - kVLag;                     // V of tile m
            if (m >= 0) {
                if (m >= 1 && !warp_wait(&mb_vempty, (m - 1) & 1, budget, abort_flag)) { fail(a.status, abort_flag, 31); break; }
                if (elect_one()) {
                    uint8_t* dst = sm + SM_V;
                    mbar_arrive_expect_tx(&mb_vfull, 16384);
                    tma_load_4d(dst, &vmap, &mb_vfull, 0, vc.h, vc.jt * kC, vc.l);
                    tma_load_4d(dst + 8192, &vmap, &mb_vfull, 64, vc.h, vc.jt * kC, vc.l);
                }
                __syncwarp();
                vp = m;
                vc.next(sch, a);
            }
        }
        if (__any_sync(0xffffffffu, *abort_flag != 0) && lane == 0) {
            // every copy this warp issued lands before the CTA ends
            for (int b = 0; b < kKSlots; ++b)
                if (kp[b] >= 0) mbar_wait(&mb_kfull[b], (kp[b] / kKSlots) & 1, budget);
            if (vp >= 0) mbar_wait(&mb_vfull, vp & 1, budget);
        }
        __syncwarp();
    } else if (warp >= kProdWarp0) {
        // =========================================================== producer: the images and decay
        // constants of every tile; group 0 (warps 8-11) the even tiles, group 1 (warps 4-7) the odd
        const int grp = warp >= 8 ? 0 : 1;
        const int pw = warp & 3;                       // 0, 1: K K^T readers (TMEM lanes 32 pw ..); 2: constants
        const int pt = pw * 32 + lane;                 // thread of the group, 0..127
        const int bar_id = kBarProd + grp;
        float* fws = reinterpret_cast<float*>(sm + SM_PW + grp * kPwBytes);
        float* Mt = fws + PW_MT;                       // rows 0..31 of diag(beta) L (columns 0..31)
        float* Mb = fws + PW_MB;                       // rows 32..63 (columns 0..63)
        float* Nt = fws + PW_NT;                       // the same rows of (I + diag(beta) L)^-1
        float* Nb = fws + PW_NB;
        float* Pm = fws + PW_P;                        // block products
        auto mrow = [&](int r) { return r < 32 ? Mt + r * kTS : Mb + (r - 32) * kBS; };
        auto nrow = [&](int r) { return r < 32 ? Nt + r * kTS : Nb + (r - 32) * kBS; };
        const int g = lane >> 2, tq = lane & 3;        // mma.sync fragment coordinates
        // cursors at the group's tile J and at J - 1 (the deferred scale before J depends on it)
        TileCursor cc, cq;
        cc.init(sch, a);
        cq = cc;
        if (grp == 1 && NJ > 1) cc.next(sch, a);
        // loads, one group-tile ahead: warp 2 the g and beta of the tile's tokens lane, 32 + lane and
        // the g of tile J - 1 when it is in J's slot; warps 0, 1 the beta of token 32 pw + lane
        struct Gb { float g0, g1, b0, b1, q0, q1; };
        auto load_gb = [&](const TileCursor& c, const TileCursor& cp, bool prev_same) {
            Gb v = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
            const int t0 = c.jt * kC + lane, t1 = t0 + 32;
            const size_t base = (size_t)c.l * a.T;
            if (pw == 2) {
                v.g0 = t0 < a.T ? a.g[(base + t0) * a.Hv + c.h] : 0.f;
                v.g1 = t1 < a.T ? a.g[(base + t1) * a.Hv + c.h] : 0.f;
                v.b0 = t0 < a.T ? a.beta[(base + t0) * a.Hv + c.h] : 0.f;
                v.b1 = t1 < a.T ? a.beta[(base + t1) * a.Hv + c.h] : 0.f;
                if (prev_same) {
                    const int s0 = cp.jt * kC + lane, s1 = s0 + 32;
                    const size_t pb = (size_t)cp.l * a.T;
                    v.q0 = s0 < a.T ? a.g[(pb + s0) * a.Hv + cp.h] : 0.f;
                    v.q1 = s1 < a.T ? a.g[(pb + s1) * a.Hv + cp.h] : 0.f;
                }
            } else if (pw < 2) {
                const int tb = t0 + 32 * pw;
                v.b0 = tb < a.T ? a.beta[(base + tb) * a.Hv + c.h] : 0.f;
            }
            return v;
        };
        // the tile's cumulative log-decay: inclusive scans of its two halves (both groups use this
        // order, so the deferred scale they compute for a tile agrees bit for bit)
        auto scan_tile = [&](float g0, float g1, float& G0, float& G1) {
            G0 = g0; G1 = g1;
#pragma unroll
            for (int m = 1; m < 32; m <<= 1) {
                const float y0 = __shfl_up_sync(0xffffffffu, G0, m);
                const float y1 = __shfl_up_sync(0xffffffffu, G1, m);
                if (lane >= m) { G0 += y0; G1 += y1; }
            }
            G1 += __shfl_sync(0xffffffffu, G0, 31);
            return __shfl_sync(0xffffffffu, G1, 31);
        };
        Gb cur = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
        if (pw < 3 && grp < NJ) {
            grid_dep_wait();
            cur = load_gb(cc, cq, grp == 1 && cq.k == cc.k);
        }
        float sig_last = 1.f;                          // sig after the group's previous tile
        bool failed = false;
        for (int J = grp; J < NJ; J += 2) {
            const int slot2 = (J >> 1) & 1;
            float* sBeta = fws + PW_BETA + 64 * slot2;
            float* sDelta = fws + PW_DELTA + 64 * slot2;
            float* sUC = fws + PW_UC + 4 * slot2;
            const bool first_of_slot = cc.jt == cc.tb;
            const bool prev_first = cq.jt == cq.tb;    // (J - 1 in J's slot only when !first_of_slot)
            const Gb now = cur;
            TileCursor nq = cc, nc = cc;               // the group's next tile J + 2 and J + 1
            if (J + 2 < NJ) {
                nq.next(sch, a);
                nc = nq;
                nc.next(sch, a);
                if (pw < 3) cur = load_gb(nc, nq, nq.k == nc.k);
            }
            DecayStep dst;
            float wn0 = 0.f, wn1 = 0.f;
            if (pw == 2) {
                // ---- constants of the tile's 64 tokens (lane: tokens lane and 32 + lane)
                float sig_b = 1.f;                     // a slot starts from the true state
                if (!first_of_slot) {                  // tile J - 1 (the other group's) in the same slot
                    float Q0, Q1;
                    const float GQ = scan_tile(now.q0, now.q1, Q0, Q1);
                    sig_b = decay_step(expf(GQ) * (prev_first ? 1.f : sig_last)).sig;
                }
                float G0, G1;
                const float GC = scan_tile(now.g0, now.g1, G0, G1);
                dst = decay_step(expf(GC) * sig_b);
                sig_last = dst.sig;
                const float d0 = expf(GC - G0), d1 = expf(GC - G1);
                sBeta[lane] = now.b0; sBeta[32 + lane] = now.b1;
                sDelta[lane] = d0; sDelta[32 + lane] = d1;
                const float ud0 = dst.u * d0, ud1 = dst.u * d1;
                wn0 = ud0 >= 0x1p-60f ? 1.f / ud0 : 0.f;   // column t of E is u delta_t u_t
                wn1 = ud1 >= 0x1p-60f ? 1.f / ud1 : 0.f;
                if (lane == 0) { sUC[0] = dst.u; sUC[1] = dst.c; }
            } else if (pw < 2) {
                // ---- rows 32 pw .. 32 pw + 31 of diag(beta) L from K K^T (warp 1: also the block
                // left of the diagonal, in full)
                const bool ok = wait_bar(&mb_kk[grp], (J >> 1) & 1, budget, abort_flag);
                if (!ok) { fail(a.status, abort_flag, 20); failed = true; }
                tc_fence_after();
                if (ok) {
                    const uint32_t base = tm + ((uint32_t)(32 * pw) << 16) + TM_KK;
                    float* row = mrow(32 * pw + lane);
                    const float bt = now.b0;
                    float kk[32];
                    tmem_ld32(base + 32 * pw, kk);         // the diagonal block
                    tmem_ld_wait();
#pragma unroll
                    for (int c4 = 0; c4 < 8; ++c4) {
                        float4 v;
                        v.x = (4 * c4 + 0 < lane) ? bt * kk[4 * c4 + 0] : 0.f;
                        v.y = (4 * c4 + 1 < lane) ? bt * kk[4 * c4 + 1] : 0.f;
                        v.z = (4 * c4 + 2 < lane) ? bt * kk[4 * c4 + 2] : 0.f;
                        v.w = (4 * c4 + 3 < lane) ? bt * kk[4 * c4 + 3] : 0.f;
                        *reinterpret_cast<float4*>(row + 32 * pw + 4 * c4) = v;
                    }
                    if (pw == 1) {                         // rows 32..63 x columns 0..31
                        tmem_ld32(base, kk);
                        tmem_ld_wait();
#pragma unroll
                        for (int c4 = 0; c4 < 8; ++c4)
                            *reinterpret_cast<float4*>(row + 4 * c4) =
                                make_float4(bt * kk[4 * c4], bt * kk[4 * c4 + 1], bt * kk[4 * c4 + 2], bt * kk[4 * c4 + 3]);
                    }
                }
                tc_fence_before();
                __syncwarp();
                if (lane == 0) mbar_arrive(&mb_kkfree);
            }
            if (named_sync_or(bar_id, kProd, failed || *abort_flag)) break;          // (1)
            if (pw < 2) {
                // the four 16 x 16 diagonal blocks of N by forward substitution, one column per lane;
                // the next row's coefficients are loaded while the current row is formed
                const int o = 32 * pw + 16 * (lane >> 4), jc = lane & 15;
                float x[16];
#pragma unroll
                for (int rr = 0; rr < 16; ++rr) x[rr] = (rr == jc) ? 1.f : 0.f;
                float4 cur4[4], nxt4[4];
                cur4[0] = *reinterpret_cast<const float4*>(mrow(o + 1) + o);
#pragma unroll
                for (int rr = 1; rr < 16; ++rr) {
                    if (rr + 1 < 16) {
#pragma unroll
                        for (int c4 = 0; c4 < 4; ++c4)
                            if (4 * c4 < rr + 1) nxt4[c4] = *reinterpret_cast<const float4*>(mrow(o + rr + 1) + o + 4 * c4);
                    }
                    float sacc[4] = {0.f, 0.f, 0.f, 0.f};     // four short FMA chains
#pragma unroll
                    for (int c4 = 0; c4 < 4; ++c4) {
                        const int c = 4 * c4;
                        if (c < rr) {
                            sacc[0] = fmaf(cur4[c4].x, x[c], sacc[0]);
                            if (c + 1 < rr) sacc[1] = fmaf(cur4[c4].y, x[c + 1], sacc[1]);
                            if (c + 2 < rr) sacc[2] = fmaf(cur4[c4].z, x[c + 2], sacc[2]);
                            if (c + 3 < rr) sacc[3] = fmaf(cur4[c4].w, x[c + 3], sacc[3]);
                        }
                    }
                    if (rr > jc) x[rr] = -((sacc[0] + sacc[1]) + (sacc[2] + sacc[3]));
#pragma unroll
                    for (int c4 = 0; c4 < 4; ++c4) cur4[c4] = nxt4[c4];
                }
#pragma unroll
                for (int rr = 0; rr < 16; ++rr) nrow(o + rr)[o + jc] = x[rr];
                if ((lane >> 4) == 0) {
#pragma unroll
                    for (int rr = 0; rr < 16; ++rr) nrow(o + rr)[o + 16 + jc] = 0.f;   // the block above
                }
            }
            if (named_sync_or(bar_id, kProd, *abort_flag)) break;                    // (2)
            {   // 16 -> 32, warp (p, nh): in 32-block p, columns 8 nh .. of
                //   P = M[16..32][0..16] N[0..16][0..16],  then  N[16..32][0..16] = -N[16..32][16..32] P
                // (tensor-core fragments, three-term bfloat16 products)
                const int p = pw >> 1, nh = pw & 1, o = 32 * p;
                const int ld = p ? kBS : kTS;
                float d[4] = {0.f, 0.f, 0.f, 0.f};
                mma_f32_split<1>(d, mrow(o + 16) + o, ld, nrow(o) + o + 8 * nh, ld, g, tq);
                float* pp = Pm + 16 * p * kPS + 8 * nh;
                *reinterpret_cast<float2*>(pp + g * kPS + 2 * tq) = make_float2(d[0], d[1]);
                *reinterpret_cast<float2*>(pp + (g + 8) * kPS + 2 * tq) = make_float2(d[2], d[3]);
                __syncwarp();
                float e[4] = {0.f, 0.f, 0.f, 0.f};
                mma_f32_split<1>(e, nrow(o + 16) + o + 16, ld, pp, kPS, g, tq);
                float* np = nrow(o + 16) + o + 8 * nh;
                *reinterpret_cast<float2*>(np + g * ld + 2 * tq) = make_float2(-e[0], -e[1]);
                *reinterpret_cast<float2*>(np + (g + 8) * ld + 2 * tq) = make_float2(-e[2], -e[3]);
            }
            if (named_sync_or(bar_id, kProd, *abort_flag)) break;                    // (3)
            {   // 32 -> 64, warp (mt, nh): rows 16 mt .., columns 16 nh .. of
                //   P = M[32..64][0..32] N[0..32][0..32],  then  N[32..64][0..32] = -N[32..64][32..64] P
                const int mt = pw >> 1, nh = pw & 1;
                float d0[4] = {0.f, 0.f, 0.f, 0.f}, d1[4] = {0.f, 0.f, 0.f, 0.f};
                mma_f32_split<2>(d0, Mb + 16 * mt * kBS, kBS, Nt + 16 * nh, kTS, g, tq);
                mma_f32_split<2>(d1, Mb + 16 * mt * kBS, kBS, Nt + 16 * nh + 8, kTS, g, tq);
                float* pp = Pm + 16 * mt * kPS + 16 * nh;
                *reinterpret_cast<float2*>(pp + g * kPS + 2 * tq) = make_float2(d0[0], d0[1]);
                *reinterpret_cast<float2*>(pp + (g + 8) * kPS + 2 * tq) = make_float2(d0[2], d0[3]);
                *reinterpret_cast<float2*>(pp + g * kPS + 8 + 2 * tq) = make_float2(d1[0], d1[1]);
                *reinterpret_cast<float2*>(pp + (g + 8) * kPS + 8 + 2 * tq) = make_float2(d1[2], d1[3]);
                if (named_sync_or(bar_id, kProd, *abort_flag)) break;                // (4)
                float e0[4] = {0.f, 0.f, 0.f, 0.f}, e1[4] = {0.f, 0.f, 0.f, 0.f};
                mma_f32_split<2>(e0, Nb + 16 * mt * kBS + 32, kBS, Pm + 16 * nh, kPS, g, tq);
                mma_f32_split<2>(e1, Nb + 16 * mt * kBS + 32, kBS, Pm + 16 * nh + 8, kPS, g, tq);
                float* np = Nb + 16 * mt * kBS + 16 * nh;
                *reinterpret_cast<float2*>(np + g * kBS + 2 * tq) = make_float2(-e0[0], -e0[1]);
                *reinterpret_cast<float2*>(np + (g + 8) * kBS + 2 * tq) = make_float2(-e0[2], -e0[3]);
                *reinterpret_cast<float2*>(np + g * kBS + 8 + 2 * tq) = make_float2(-e1[0], -e1[1]);
                *reinterpret_cast<float2*>(np + (g + 8) * kBS + 8 + 2 * tq) = make_float2(-e1[2], -e1[3]);
            }
            // the images are free once the products of tile J - 1 (the other group's) have completed,
            // the constants slot once the chain has read those of tile J - 2
            if (J >= 1 && !wait_bar(&mb_bfree[(J - 1) & 1], ((J - 1) >> 1) & 1, budget, abort_flag)) {
                fail(a.status, abort_flag, 21); failed = true;
            }
            if (J >= 2 && !wait_bar(&mb_iempty[J & 1], ((J >> 1) - 1) & 1, budget, abort_flag)) {
                fail(a.status, abort_flag, 22); failed = true;
            }
            if (named_sync_or(bar_id, kProd, failed || *abort_flag)) break;          // (5)
            {   // images: row t = pt / 2, columns 32 hh .. 32 hh + 31 of N_beta = N diag(beta) (zero
                // above the diagonal)
                const int t = pt >> 1, hh = pt & 1;
                const float u = sUC[0];
                uint8_t* b1 = sm + SM_B1;
                uint8_t* b3 = sm + SM_B3;
                const bool zero_half = t < 32 && hh == 1;
                const float* nr = nrow(t) + (zero_half ? 0 : 32 * hh);
#pragma unroll 1
                for (int g8 = 0; g8 < 4; ++g8) {        // 8 columns (one 16-byte chunk of bf16) at a time
                    const int c = 32 * hh + 8 * g8;
                    uint32_t h3[4] = {0u, 0u, 0u, 0u}, l3[4] = {0u, 0u, 0u, 0u};
                    uint32_t h1[4] = {0u, 0u, 0u, 0u}, l1[4] = {0u, 0u, 0u, 0u};
                    if (!zero_half) {
                        const float4 n0 = *reinterpret_cast<const float4*>(nr + 8 * g8);
                        const float4 n1 = *reinterpret_cast<const float4*>(nr + 8 * g8 + 4);
                        const float4 bv0 = *reinterpret_cast<const float4*>(sBeta + c);
                        const float4 bv1 = *reinterpret_cast<const float4*>(sBeta + c + 4);
                        const float4 dv0 = *reinterpret_cast<const float4*>(sDelta + c);
                        const float4 dv1 = *reinterpret_cast<const float4*>(sDelta + c + 4);
                        const float nv[8] = {n0.x, n0.y, n0.z, n0.w, n1.x, n1.y, n1.z, n1.w};
                        const float bv[8] = {bv0.x, bv0.y, bv0.z, bv0.w, bv1.x, bv1.y, bv1.z, bv1.w};
                        const float dv[8] = {dv0.x, dv0.y, dv0.z, dv0.w, dv1.x, dv1.y, dv1.z, dv1.w};
                        float nb[8], w1[8];
#pragma unroll
                        for (int i = 0; i < 8; ++i) {
                            nb[i] = (c + i <= t) ? nv[i] * bv[i] : 0.f;
                            w1[i] = u * nb[i] * dv[i];
                        }
#pragma unroll
                        for (int i = 0; i < 4; ++i) {
                            split2(nb[2 * i], nb[2 * i + 1], h3[i], l3[i]);
                            split2(w1[2 * i], w1[2 * i + 1], h1[i], l1[i]);
                        }
                    }
                    const uint32_t off = sw128_offset(t, c >> 3);
                    *reinterpret_cast<uint4*>(b3 + off) = make_uint4(h3[0], h3[1], h3[2], h3[3]);
                    *reinterpret_cast<uint4*>(b3 + 8192 + off) = make_uint4(l3[0], l3[1], l3[2], l3[3]);
                    *reinterpret_cast<uint4*>(b1 + off) = make_uint4(h1[0], h1[1], h1[2], h1[3]);
                    *reinterpret_cast<uint4*>(b1 + 8192 + off) = make_uint4(l1[0], l1[1], l1[2], l1[3]);
                }
            }
            if (pw == 2) {                              // the chain's and the MMA's constants
                float* cs = cst + (J & 1) * kConstWords;
                cs[lane] = wn0;
                cs[32 + lane] = wn1;
                if (lane == 0) {
                    cs[64] = dst.sig;
                    cs[65] = dst.pass;
                    reinterpret_cast<int*>(cs)[66] = dst.shift;
                    cs[67] = dst.c;
                }
            }
            fence_async_smem();                         // generic writes -> the tensor core's reads
            __syncwarp();
            if (lane == 0) mbar_arrive(&mb_ifull[J & 1]);
            cq = nq;
            cc = nc;
        }
    } else {
        // =========================================================== state chain (warps 0-3)
        const int q = warp;                              // TMEM lane quadrant
        const int r = 32 * q + lane;                     // row of S (value index)
        const uint32_t lane_off = (uint32_t)(32 * q) << 16;
        TileCursor cc;
        cc.init(sch, a);
        // W(jj) = -c Q^T in tf32: this thread's d_k row c = r of Q, tokens 0..63, into rows t of the
        // K-major W (column block q, its 4-byte slot of row t).  Q(jj) is complete and W's last
        // reader, E(jj-1) += S~ W(jj-1), has completed.
        auto make_w = [&](int jj) -> bool {
            bool ok = wait_bar(&mb_q, jj & 1, budget, abort_flag);
            ok = wait_bar(&mb_ifull[jj & 1], (jj >> 1) & 1, budget, abort_flag) && ok;
            tc_fence_after();
            const float cneg = -cst[(jj & 1) * kConstWords + 67];
            uint8_t* wb = sm + SM_W + q * 8192 + (lane & 3) * 4;
            const int chunk = lane >> 2;
#pragma unroll 1
            for (int hh = 0; hh < 2; ++hh) {
                float qv[32];
                tmem_ld32(tm + lane_off + TM_Q + 32 * hh, qv);
                tmem_ld_wait();
#pragma unroll
                for (int i = 0; i < 32; ++i)
                    *reinterpret_cast<uint32_t*>(wb + sw128_offset(32 * hh + i, chunk)) = to_tf32(cneg * qv[i]);
            }
            fence_async_smem();
            tc_fence_before();
            return ok;
        };
        // a slot's starting state (from the state or hand-over entry i - 1) into TMEM as S~ and
        // S_before; `den` gets this thread's sum of squares
        auto install = [&](int slot, float& den) -> bool {
            int lh, tb, te;
            sch.slot(slot, a.n_tiles, lh, tb, te);
            const bool from_ho = sch.is_suffix(slot);
            bool ok = true;
            if (from_ho) {                               // one thread waits for CTA i - 1's state
                if (tid == 0) {
                    const uint32_t bit = 1u << ((me - 1) & 31);
                    uint32_t* w = bits_state + ((me - 1) >> 5);
                    const uint64_t t0 = global_ns();
                    while ((ld_acquire(w) & bit) == 0) {
                        if (*abort_flag || global_ns() - t0 > budget) { fail(a.status, abort_flag, 42); break; }
                        __nanosleep(64);
                    }
                    atomicAnd(w, ~bit);                  // consumed: zero for the next call
                }
                ok = !named_sync_or(kBarChain, kChain, *abort_flag);
            }
            const float* src = (from_ho ? a.ho_state + (size_t)(me - 1) * kD * kD : a.state + (size_t)lh * kD * kD)
                               + (size_t)r * kD;
            den = 0.f;
            if (ok) {
#pragma unroll 1
                for (int g8 = 0; g8 < 8; ++g8) {
                    float v[16];
                    ld16_global(src + 16 * g8, v, from_ho);
                    uint32_t u32[16];
#pragma unroll
                    for (int e = 0; e < 16; ++e) { den = fmaf(v[e], v[e], den); u32[e] = __float_as_uint(v[e]); }
                    tmem_st16(tm + lane_off + TM_S + 16 * g8, u32);
                    tmem_st16(tm + lane_off + TM_SB + 16 * g8, u32);
                }
            }
            return ok;
        };
        float den = 0.f, sig = 1.f;
        // Write sizes (optional): column t of E is u delta_t u_t, u_t = beta_t (v_t - alpha_t S_{t-1}
        // k_t) the token's write.  The pass sums each column's squares over the warp's 32 rows,
        // rescales them by the constant (1 / (u delta_t))^2 and adds them into s_u2 (four warps per
        // column); at the next tile warp 0 takes the square roots and sums them into the head's total.
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
                sum += __ldcg(a.ho_wsum + me - 1);
                atomicAnd(w, ~bit);
            }
            a.wnorm[lh] = sum;
            return true;
        };
        auto fold_writes = [&](int jj) {                   // warp 0: tile jj's sizes into wacc
            float* b = s_u2[jj & 1];
            float sacc = sqrtf(b[lane]) + sqrtf(b[32 + lane]);
            b[lane] = 0.f;
            b[32 + lane] = 0.f;
#pragma unroll
            for (int m = 16; m >= 1; m >>= 1) sacc += __shfl_xor_sync(0xffffffffu, sacc, m);
            wacc += sacc;
        };
        bool stop = NJ == 0;
        if (!stop) {
            // ---- the CTA's first slot: its state into TMEM, and W of its first tile
            bool ok = install(0, den);
            ok = make_w(0) && ok;
            tmem_st_wait();
            tc_fence_before();
            if (!ok) fail(a.status, abort_flag, 14);
            warp_arrive(&mb_ready, lane);
        }
        for (int j = 0; j < NJ && !stop; ++j) {
            const int lh = cc.lh, slot = cc.k;
            const bool last = cc.jt == cc.te - 1;          // the slot's last tile
            if (named_sync_or(kBarChain, kChain, *abort_flag)) break;
            if (want_w && j > 0 && warp == 0) {
                fold_writes(j - 1);
                if (prev_last) {
                    if (lane == 0 && !put_wsum(prev_slot, prev_lh, wacc)) fail(a.status, abort_flag, 44);
                    wacc = 0.f;
                }
            }
            // ---- E(j) is complete (and E += S~ W has read the state and W)
            if (!wait_bar(&mb_u, j & 1, budget, abort_flag)) fail(a.status, abort_flag, 10);
            tc_fence_after();
            const float* cs = cst + (j & 1) * kConstWords;
            const float pass_f = cs[65];
            const float sig_after = cs[64];
            if (pass_f >= 0.f) {
                // the decay would take the deferred scale out of range: S~ <- p S~ (the state
                // update of this tile has not been issued: it waits for this pass)
#pragma unroll 1
                for (int g8 = 0; g8 < 8; ++g8) {
                    float sv[16];
                    tmem_ld16(tm + lane_off + TM_S + 16 * g8, sv);
                    tmem_ld_wait();
                    uint32_t su[16];
#pragma unroll
                    for (int e = 0; e < 16; ++e) su[e] = __float_as_uint(sv[e] * pass_f);
                    tmem_st16(tm + lane_off + TM_S + 16 * g8, su);
                }
            }
#pragma unroll 1
            for (int hh = 0; hh < 2; ++hh) {
                // ---- pass: 32 token columns of E -> (hi, lo) A operand, in place
                const uint32_t eb = tm + lane_off + TM_E + (j & 1) * 64 + 32 * hh;
                float e[32];
                tmem_ld32(eb, e);
                tmem_ld_wait();
                if (want_w) {
                    // squares summed over the warp's 32 rows, column by column: halving exchanges
                    // leave lane c with column c
                    const float wf = cs[32 * hh + lane];
                    float x[32];
#pragma unroll
                    for (int i = 0; i < 32; ++i) x[i] = e[i] * e[i];
#pragma unroll
                    for (int w = 16; w >= 1; w >>= 1) {
                        const bool up = (lane & w) != 0;
#pragma unroll
                        for (int i = 0; i < w; ++i) {
                            const float send = up ? x[i] : x[i + w];
                            x[i] = (up ? x[i + w] : x[i]) + __shfl_xor_sync(0xffffffffu, send, w);
                        }
                    }
                    atomicAdd(&s_u2[j & 1][32 * hh + lane], x[0] * wf * wf);
                }
                uint32_t hi[16], lo[16];
#pragma unroll
                for (int i = 0; i < 16; ++i) split2(e[2 * i], e[2 * i + 1], hi[i], lo[i]);
                tmem_st16(eb, hi);
                tmem_st16(eb + 16, lo);
            }
            tmem_st_wait();
            tc_fence_before();
            warp_arrive(&mb_uready, lane);
            warp_arrive(&mb_iempty[j & 1], lane);          // the tile's constants are read
            sig = sig_after;
            // ---- while the state update runs: W of the next tile
            const bool has_next = j + 1 < NJ;
            bool ok = true;
            if (has_next) ok = make_w(j + 1);
            if (!ok) fail(a.status, abort_flag, 15);
            if (last) {
                // ---- slot boundary: S_after = sig S~ out, drift partials against S_before, the next
                // slot's state in
                const bool prefix = sch.is_prefix(slot);
                const bool shared_end = sch.is_suffix(slot);   // S_before: the head's stored state
                if (!wait_bar(&mb_s, j & 1, budget, abort_flag)) { fail(a.status, abort_flag, 12); ok = false; }
                tc_fence_after();
                float num = 0.f, den_end = 0.f;
                float* dstp = (prefix ? a.ho_state + (size_t)me * kD * kD : a.state + (size_t)lh * kD * kD)
                              + (size_t)r * kD;
                const float* sbp = a.state + (size_t)lh * kD * kD + (size_t)r * kD;
                if (ok) {
#pragma unroll 1
                    for (int g8 = 0; g8 < 8; ++g8) {
                        float sa[16], sb[16];
                        tmem_ld16(tm + lane_off + TM_S + 16 * g8, sa);
                        if (shared_end) {
                            ld16_global(sbp + 16 * g8, sb, true);
#pragma unroll
                            for (int e = 0; e < 16; ++e) den_end = fmaf(sb[e], sb[e], den_end);
                        } else {
                            tmem_ld16(tm + lane_off + TM_SB + 16 * g8, sb);
                        }
                        tmem_ld_wait();
#pragma unroll
                        for (int e = 0; e < 16; ++e) {
                            sa[e] *= sig;
                            const float d = sa[e] - sb[e];
                            num = fmaf(d, d, num);
                        }
                        float4* o4 = reinterpret_cast<float4*>(dstp + 16 * g8);
#pragma unroll
                        for (int e = 0; e < 4; ++e) o4[e] = make_float4(sa[4 * e], sa[4 * e + 1], sa[4 * e + 2], sa[4 * e + 3]);
                    }
                }
                // partial sums: pairwise in fp32, over the warp's lanes and then over the warps
                float fn = num, fd = shared_end ? den_end : den;
#pragma unroll
                for (int m = 16; m >= 1; m >>= 1) {
                    fn += __shfl_xor_sync(0xffffffffu, fn, m);
                    fd += __shfl_xor_sync(0xffffffffu, fd, m);
                }
                if (lane == 0) { s_red[0][warp] = fn; s_red[1][warp] = fd; }
                if (prefix) __threadfence();                  // the hand-over state is in memory ...
                if (named_sync_or(kBarChain, kChain, !ok || *abort_flag)) { stop = true; break; }
                if (prefix && tid == 0) atomicOr(bits_state + (me >> 5), 1u << (me & 31));   // ... before CTA i + 1 reads it
                if (warp == 0 && a.partials != nullptr && !prefix) {   // a shared head: at its end
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
                if (has_next) {
                    if (!install(slot + 1, den)) fail(a.status, abort_flag, 16);
                    tmem_st_wait();
                }
                sig = 1.f;
            }
            if (has_next) {
                tc_fence_before();
                warp_arrive(&mb_ready, lane);               // W(j + 1) (and a new slot's state) ready
            }
            prev_lh = lh;
            prev_slot = slot;
            prev_last = last;
            cc.next(sch, a);
        }
        // the CTA's last tile (always a slot's last) once every warp's pass has added to it
        if (want_w && NJ > 0 && !named_sync_or(kBarChain, kChain, *abort_flag) && warp == 0) {
            fold_writes(NJ - 1);
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
    CUtensorMap kmap, vmap;
    if (!make_map(&kmap, a.k, a.L, a.T, a.Hk) || !make_map(&vmap, a.v, a.L, a.T, a.Hv)) return cudaErrorInvalidValue;
    // The attribute is per device; setting it on every launch costs little and stays correct after
    // a device reset and from any host thread.
    cudaError_t e = cudaFuncSetAttribute(gdn_fused_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         (int)kSmemAlloc);
    if (e != cudaSuccess) return e;
    const int n_tiles = (a.T + kC - 1) / kC;
    TcArgs t;
    t.L = a.L; t.Hk = a.Hk; t.Hv = a.Hv; t.T = a.T; t.n_tiles = n_tiles;
    t.g = a.g; t.beta = a.beta;
    t.state = a.state; t.partials = a.partials; t.wnorm = a.wnorm; t.status = a.status;
    t.ho_bits = reinterpret_cast<uint32_t*>(a.status) + 4;
    t.ho_state = reinterpret_cast<float*>(a.scratch + sl.ho_state);
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
        e = cudaLaunchKernelEx(&cfg, gdn_fused_kernel, kmap, vmap, t);
        if (e != cudaErrorCooperativeLaunchTooLarge) return e;
        (void)cudaGetLastError();                 // fewer SMs than the grid: whole heads instead
        t.split = 0;
    }
    cfg.attrs = nullptr;
    cfg.numAttrs = 0;
    return cudaLaunchKernelEx(&cfg, gdn_fused_kernel, kmap, vmap, t);
}

}  // namespace deltas
