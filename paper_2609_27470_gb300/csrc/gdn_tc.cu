// Gated delta rule over one chunk on the Blackwell tensor cores (tcgen05 + TMEM + TMA), d = 128,
// bfloat16 k/v, fp32 state, with the state-drift partials fused in.
//
// Paper: Sec. 3.2, Eq. 1/2 (the recurrence) and Eq. 3 (drift numerator / denominator per layer
// and head).  The chunk is processed in tiles of C = 64 tokens with the chunkwise (WY) form of
// Eq. 1: with G the inclusive cumulative log-decay inside the tile, gamma = exp(G),
//   A[t][i] = beta_t exp(G_t - G_i) k_t.k_i  (i < t),   T = (I + A)^-1 diag(beta),
//   X = K S0^T,   W = V - diag(gamma) X,   U = T W,
//   S_C = gamma_C S0 + U~^T K,   U~[t] = exp(G_C - G_t) U[t].
// Padded tokens of a ragged last tile carry k = v = 0, g = 0, beta = 0 and change nothing.
//
// Two kernels.  T and the tile's decay constants depend on k, g and beta only, so the factor
// kernel builds them for every (layer, value head, tile) at once, several CTAs per SM, and writes
// one record per tile into the workspace: T~ = diag(exp(G_C - G)) T as the bfloat16 (hi, lo) pair
// in the swizzled layout the tensor core reads, -gamma and gamma_C.  The update kernel then runs
// the part that is sequential in the tiles, the state chain, with nothing else on the SM.
//
// Update kernel: one persistent CTA per SM takes (layer, value head) pairs in turn, or equal runs
// of tiles with a head at each run boundary split between two CTAs, or, with few heads, two
// segments of each head on three CTAs (see ChainSched); the tiles of its slots form one pipeline.
// With the read-out a third kernel (gdn_readout_kernel) forms the outputs.  A head's state lives in TMEM from its first tile to its last
// (S_before beside it, for the drift), so the state is read from and written to HBM exactly once;
// the next head's state is loaded into shared memory while the current head runs, and the head
// boundary swaps the two in one pass that also forms the drift partials.  Per tile:
//   V region  <- V^T                       (MMA: V tile times an identity matrix, exact)
//   X region  <- S~ K^T                     (tf32 MMA, K exact in fp32)
//   W pass:   W^T = V^T - sig X diag(gamma), x u_scale -> (hi, lo) in place over X   (chain)
//   U region  <- W^T T~^T = U~^T / ...      (MMA)
//   U~ pass:  -> (hi, lo) in place                          (chain)
//   S~        += U~^T K                     (MMA)
// so the chain's passes are a few loads, an FMA, a split and a store per element, and the
// per-token decays ride on the W pass and on T~.
//
// Precision.  Keys and values are exact in bfloat16.  The state never leaves fp32 inside the
// tile loop: TMEM holds S~ with S = sig S~, and X reads S~ straight from TMEM as the A operand of
// a kind::tf32 product; the hardware keeps 10 mantissa bits of S~ (a relative error below 2^-10
// per element) while K is exact, an error that reaches the state only through the
// delta correction and decay with it (a CPU simulation of the truncation gives a state error vs
// fp64 of ~2e-4 at the slowest decay the inputs use, 5e-6 at a typical one).  The other products
// take a two-term bfloat16 split (x = hi + lo, hi = bf16(x), lo = bf16(x - hi)) of each fp32
// operand:
//   V^T I                           exact                                        1 MMA group
//   X^T  = S~ K^T                   S~ (tf32, from TMEM) K (exact in tf32)       1 MMA group
//   U~^T = W^T T~^T                  Whi T~hi + Whi T~lo + Wlo T~hi                3 MMA groups
//   S   += U~^T K                   (U~hi + U~lo) K                              2 MMA groups
//   K K^T (factor kernel)           exact inputs                                 1 MMA group
// All products accumulate in fp32 in TMEM.
//
// Deferred decay: the tile decay gamma_C is folded into the scalar sig instead of a pass that
// multiplies S by gamma_C; the W pass applies sig and scales W by u_scale = 1 / (gamma_C sig) so that
// MMA_S adds onto S~ directly.  When sig gamma_C would fall below 2^-30 the tile writes
// gamma_C sig S~ back into TMEM and sig restarts at 1 (u_scale = 1), so 1 / sig stays far from the
// fp32 range limit.  The head's last tile multiplies by sig when it reads the state out.
//
// Update-kernel warp roles (19 warps):
//   0-15  state chain: warp w serves TMEM lanes 32 (w % 4) .. + 31 (state rows) and column group
//         w / 4; per tile the W and U~ passes (16 token columns each) and the next tile's K in
//         fp32 (two 16-byte chunks each), at head boundaries the state swap and the drift partials
//   16    TMEM allocation and every tcgen05.mma (one elected lane issues; the warp stays
//         converged); it also releases the input buffers by tcgen05.commit
//   17    tile loads: K, V (TMA) and the WY records (bulk copy), as buffers are released
//   18    state moves: each head's state into the staging buffer, S_after out of it
// A TMA or bulk copy occupies the issuing thread for a time that grows with its size, so no copy
// is issued from a role on the chain's critical path.  Roles hand work to each other through
// mbarriers only.  Every wait is bounded; a wait that runs out records DELTAS_ERR_TIMEOUT, raises
// a CTA-wide abort flag so the other roles stop waiting, and the CTA drains its MMAs and copies
// before freeing TMEM.
// TMEM (512 columns, M = 128 lanes = d_v): S~ [0,128), S_before [128,256), X [256,320) (X, then
// W hi / lo packed in place), U [320,384) (likewise U~), V^T [384,448); [448,512) unused.
#include <algorithm>
#include <cmath>

#include "internal.cuh"
#include "tc_ptx.cuh"

namespace deltas {
namespace {

using namespace tc;

constexpr int kC = 64;                 // tokens per tile
constexpr int kD = 128;                // head dim (d_k = d_v)
constexpr float kLog2e = 1.4426950408889634f;
constexpr float kSigMin = 9.313225746154785e-10f;   // 2^-30: smallest deferred decay of the state

// ---- WY record of one (layer, value head, tile), written by the factor kernel, read by the update
// kernel with one bulk copy:
//   [0, 8192)       T~ hi: bfloat16 [64 t][64 i], 128-byte rows, 128-byte swizzle (K-major B operand)
//   [8192, 16384)   T~ lo, same layout
//   [16384, 16656)  float: -gamma[64], gamma_C, 3 unused
// With the read-out the record holds T itself (no row decay) and, after the constants above,
//   [16656, 16912)  float: exp(G_C - G_t)[64], the row decays, applied by the update kernel
// so that the update kernel sees each token's write u_t undecayed.
constexpr uint32_t kRecT = 16384;
constexpr uint32_t kRecConsts = 68;
constexpr uint32_t kRecBytes = kRecT + kRecConsts * 4;
constexpr uint32_t kRecBytesOut = kRecBytes + kC * 4;
static_assert(kRecBytes % 16 == 0 && kRecBytesOut % 16 == 0, "records are bulk-copied: 16-byte multiples");
__host__ __device__ constexpr uint32_t rec_bytes(bool out) { return out ? kRecBytesOut : kRecBytes; }

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

// D (16 x 8) += A (16 x 16, row) B (16 x 8, col) on the warp's tensor-core path, bf16 in, fp32
// accumulate.  Fragments (g = lane / 4, t = lane % 4), each register a bf16 pair, lower k in the
// low half: a = A[g][2t..], A[g+8][2t..], A[g][2t+8..], A[g+8][2t+8..]; b = B[2t..][g],
// B[2t+8..][g]; d as for the tf32 form.
__device__ __forceinline__ void mma_m16n8k16_bf16(float (&d)[4], const uint32_t (&a)[4], const uint32_t (&b)[2]) {
    asm volatile("mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, "
                 "{%0,%1,%2,%3};"
                 : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
                 : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b[0]), "r"(b[1]));
}

// Operands stored split: row r of A is at A + r * as (32-bit words), its word p the bf16 pair of
// hi = bf16(x) for columns (2p, 2p+1) and word a_lo + p the pair of lo = bf16(x - hi); likewise B,
// stored n-major (row n of B's storage holds column n of B).  D (16 x 8) += A[r0 .. r0+15][0..16K)
// B[0..16K)[n0 .. n0+7] over the three products lo*hi + hi*lo + hi*hi.
template <int KSTEPS>
__device__ __forceinline__ void mma_split_bf16(float (&d)[4], const uint32_t* A, int as, int a_lo, int r0,
                                               const uint32_t* B, int bs, int b_lo, int n0, int lane) {
    const int g = lane >> 2, t = lane & 3;
    const uint32_t* a0 = A + (r0 + g) * as;
    const uint32_t* a1 = A + (r0 + g + 8) * as;
    const uint32_t* b0 = B + (n0 + g) * bs;
#pragma unroll
    for (int ks = 0; ks < KSTEPS; ++ks) {
        const int p0 = 8 * ks + t, p1 = p0 + 4;
        const uint32_t ah[4] = {a0[p0], a1[p0], a0[p1], a1[p1]};
        const uint32_t al[4] = {a0[a_lo + p0], a1[a_lo + p0], a0[a_lo + p1], a1[a_lo + p1]};
        const uint32_t bh[2] = {b0[p0], b0[p1]};
        const uint32_t bl[2] = {b0[b_lo + p0], b0[b_lo + p1]};
        mma_m16n8k16_bf16(d, al, bh);
        mma_m16n8k16_bf16(d, ah, bl);
        mma_m16n8k16_bf16(d, ah, bh);
    }
}

// One element of a split row (see mma_split_bf16): hi / lo halfwords of column k; lo words start
// lo_words after the row's first word.
__device__ __forceinline__ void put_split(uint32_t* row, int k, float x, int lo_words = 16) {
    const __nv_bfloat16 h = __float2bfloat16_rn(x);
    const __nv_bfloat16 l = __float2bfloat16_rn(x - __bfloat162float(h));
    reinterpret_cast<__nv_bfloat16*>(row)[k] = h;
    reinterpret_cast<__nv_bfloat16*>(row + lo_words)[k] = l;
}

// 16 consecutive values -> split row of a 16-column operand (words 0..7 hi, 8..15 lo)
__device__ __forceinline__ void put_split16(uint32_t* row, const float* x) {
    uint32_t h[8], l[8];
#pragma unroll
    for (int i = 0; i < 8; ++i) split2(x[2 * i], x[2 * i + 1], h[i], l[i]);
    *reinterpret_cast<uint4*>(row) = make_uint4(h[0], h[1], h[2], h[3]);
    *reinterpret_cast<uint4*>(row + 4) = make_uint4(h[4], h[5], h[6], h[7]);
    *reinterpret_cast<uint4*>(row + 8) = make_uint4(l[0], l[1], l[2], l[3]);
    *reinterpret_cast<uint4*>(row + 12) = make_uint4(l[4], l[5], l[6], l[7]);
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


// shared-memory descriptor advanced by `bytes` (the start address field counts 16-byte units)
__device__ __forceinline__ uint64_t dadd(uint64_t desc, uint32_t bytes) { return desc + (uint64_t)(bytes >> 4); }

// =============================================================================================
// Factor kernel: T~ = diag(exp(G_C - G)) (I + A)^-1 diag(beta) and the decay constants of every tile
// =============================================================================================
constexpr int kWyThreads = 256;
constexpr int kWyCtasPerSm = 4;
constexpr uint32_t kWyTmemCols = 64;
constexpr int FA_S = 68;               // fp32 row stride of A: 16-byte rows; a 16-byte access by 8 threads
                                       // of 8 consecutive rows hits 8 distinct bank groups
constexpr int FX_S = 68;               // fp32 row stride of X = (I + A)^-1 (16-byte aligned rows)
// shared-memory map (bytes from a 1024-aligned base)
constexpr uint32_t WY_FA = 0;                         // fp32 [64][FA_S].  Its two 32 x 32 quarters that are
                                                      // never read as fp32 hold split operands of level 2:
                                                      // rows 32..63 x cols 0..31 = A21 (row-major), rows
                                                      // 0..31 x cols 32..63 = X11 stored n-major
constexpr uint32_t WY_K = WY_FA;                      // the next item's K tile (2 column blocks (d 0-63,
                                                      // 64-127) x 64 rows x 128 B) lands over A once level 2
                                                      // has read it; the M = 128 product of K K^T reads the
                                                      // 8 KB past the tile as rows 64..127 (output ignored)
constexpr uint32_t WY_FX = WY_FA + 64 * FA_S * 4;     // fp32 [64][FX_S]; rows 0..31 x cols 32..63 (the zero
                                                      // upper quarter) hold X22 split, row-major
constexpr uint32_t WY_TMP = WY_FX + 64 * FX_S * 4;    // level 1 products (fp32), then level 2's P split,
                                                      // n-major, rows of 36 words
constexpr uint32_t WY_L1 = WY_TMP + 32 * 36 * 4;      // level-1 split operands, 6 x 16 rows of 20 words: A10,
                                                      // A32, X11' (row-major), X22' (n-major), P1 for p = 0, 1
constexpr int kL1S = 20;                              // row stride (words): fragment loads hit distinct banks
constexpr uint32_t WY_TG = WY_L1 + 6 * 16 * kL1S * 4; // 2 buffers (item parity) x (G2[64], beta[64], row[64],
                                                      // col[64], del[64], flag)
constexpr uint32_t kTgFloats = 324;
constexpr uint32_t WY_BYTES = WY_TG + 2 * kTgFloats * 4;
constexpr uint32_t kWySmemAlloc = WY_BYTES + 1024;
static_assert(WY_TG % 16 == 0 && (kTgFloats * 4) % 16 == 0, "tile factors must be 16-byte aligned");
static_assert(kWyCtasPerSm * (kWySmemAlloc + 1024) <= 233472, "factor kernel: CTAs per SM");

struct WyArgs {
    int L, Hk, Hv, T, n_tiles;
    int out;                   // records for the read-out: T and the row decays (see the record)
    const float* g;
    const float* beta;
    uint8_t* rec;              // [L * Hv][n_tiles] records of rec_bytes(out)
    int32_t* status;
    int32_t* ho_flags;         // the update kernel's hand-over flags, reset here for this call
    int n_ho_flags;
};

__global__ void __launch_bounds__(kWyThreads, kWyCtasPerSm)
gdn_wy_kernel(const __grid_constant__ CUtensorMap kmap, WyArgs a)
{
    extern __shared__ uint8_t smem_raw[];
    uint8_t* sm = smem_raw + ((1024 - (smem_u32(smem_raw) & 1023)) & 1023);
    __shared__ uint64_t mb_k, mb_kk;
    __shared__ uint32_t s_tmem;
    __shared__ int s_fail;
    grid_dep_launch();                                // the update kernel may take SMs as they free up
    // the update kernel reads its hand-over flags only after this kernel has completed
    if (blockIdx.x == 0)
        for (int e = (int)threadIdx.x; e < a.n_ho_flags; e += kWyThreads) a.ho_flags[e] = 0;
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int n = a.n_tiles;
    const int items = a.L * a.Hv * n;                 // item = (layer * Hv + head) * n + tile
    // The workspace's wait budget bounds the CTA's first wait; the later ones keep the fixed bound
    // (a bound read at run time in every wait of these latency-bound kernels measured slower).
    const uint64_t budget0 = wait_budget_ns(a.status);
    float* fA = reinterpret_cast<float*>(sm + WY_FA);
    float* fX = reinterpret_cast<float*>(sm + WY_FX);
    float* fT = reinterpret_cast<float*>(sm + WY_TMP);
    // split level-2 operands (see the shared-memory map), row strides in 32-bit words
    uint32_t* sA21 = reinterpret_cast<uint32_t*>(fA + 32 * FA_S);        // A[32 + r][k]
    uint32_t* sX11 = reinterpret_cast<uint32_t*>(fA + 32);               // row n: X[k][n], k < 32
    uint32_t* sX22 = reinterpret_cast<uint32_t*>(fX + 32);               // row r: X[32 + r][32 + k]
    uint32_t* sP = reinterpret_cast<uint32_t*>(fT);                      // row n: P[k][n]
    constexpr int kPS = 36;
    // split level-1 operands: 16 x 16 blocks, rows of kL1S words (hi words 0..7, lo words 8..15)
    uint32_t* sL1 = reinterpret_cast<uint32_t*>(sm + WY_L1);
    uint32_t* sA10 = sL1;                                                 // A[16 + r][k]
    uint32_t* sA32 = sL1 + 16 * kL1S;                                     // A[48 + r][32 + k]
    uint32_t* sX11r = sL1 + 32 * kL1S;                                    // X[16 + r][16 + k]
    uint32_t* sX22n = sL1 + 48 * kL1S;                                    // row n: X[32 + k][32 + n]
    uint32_t* sP1 = sL1 + 64 * kL1S;                                      // p: row n of P1_p, 16 rows each

    if (warp == 0) { tmem_alloc(&s_tmem, kWyTmemCols); tmem_relinquish(); }
    if (tid == 0) {
        mbar_init(&mb_k, 1); mbar_init(&mb_kk, 1);
        fence_barrier_init();
        prefetch_tensormap(&kmap);
        s_fail = 0;
    }
    // The strictly upper 16 x 16 blocks of X are never written; zeros there let every level run
    // fixed-length (unrolled) loops over the triangular factors.
    for (int e = tid; e < 64 * FX_S; e += kWyThreads) { fX[e] = 0.f; fA[e] = 0.f; }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tm = s_tmem;

    // Items are taken in reverse record order: the records written last, still in L2 when this
    // kernel ends, are the ones of the lowest heads, which the update kernel reads first.
    auto rec_of = [&](int it) { return items - 1 - it; };
    auto item_pos = [&](int it, int& l, int& h, int& jt) {
        const int r = rec_of(it), lh = r / n;
        jt = r - lh * n; l = lh / a.Hv; h = lh - l * a.Hv;
    };
    int nk = 0, nkk = 0;                               // K loads (thread 0) / K K^T products (warp 0) issued
    auto load_k = [&](int it) {                        // thread 0: the item's K tile
        int l, h, jt;
        item_pos(it, l, h, jt);
        ++nk;
        const int kh = (int)(((long long)h * a.Hk) / a.Hv);
        mbar_arrive_expect_tx(&mb_k, 16384);
        tma_load_4d(sm + WY_K, &kmap, &mb_k, 0, kh, jt * kC, l);
        tma_load_4d(sm + WY_K + 8192, &kmap, &mb_k, 64, kh, jt * kC, l);
    };
    // g and beta of an item's 64 tokens, two per lane of warp 7, loaded one item ahead of use
    float pg[2] = {0.f, 0.f}, pb[2] = {0.f, 0.f};
    auto load_gb = [&](int it) {
        int l, h, jt;
        item_pos(it, l, h, jt);
#pragma unroll
        for (int e = 0; e < 2; ++e) {
            const int t = jt * kC + 2 * lane + e;
            const size_t gi = ((size_t)l * a.T + t) * a.Hv + h;
            pg[e] = t < a.T ? a.g[gi] : 0.f;
            pb[e] = t < a.T ? a.beta[gi] : 0.f;
        }
    };
    // Decay constants of an item from the loaded g, beta (warp 7): the update kernel's -gamma and
    // gamma_C into the record, and this kernel's G2, beta, row and column factors and
    // exp(G_C - G) into buffer `buf`.
    auto tile_constants = [&](int it, int buf) {
        float incl = pg[0] + pg[1];
#pragma unroll
        for (int m = 1; m < 32; m <<= 1) {
            const float y = __shfl_up_sync(0xffffffffu, incl, m);
            if (lane >= m) incl += y;
        }
        const float G0 = incl - pg[1], G1 = incl;
        const float GC = __shfl_sync(0xffffffffu, incl, 31);
        float* rc = reinterpret_cast<float*>(a.rec + (size_t)rec_of(it) * rec_bytes(a.out) + kRecT);
        *reinterpret_cast<float2*>(rc + 2 * lane) = make_float2(-expf(G0), -expf(G1));
        if (lane == 0) *reinterpret_cast<float4*>(rc + 64) = make_float4(expf(GC), 0.f, 0.f, 0.f);
        if (a.out) *reinterpret_cast<float2*>(rc + kRecConsts + 2 * lane) = make_float2(expf(GC - G0), expf(GC - G1));
        const float g20 = G0 * kLog2e, g21 = G1 * kLog2e;
        float lo2 = fminf(g20, g21), hi2 = fmaxf(g20, g21);
#pragma unroll
        for (int m = 16; m >= 1; m >>= 1) {
            lo2 = fminf(lo2, __shfl_xor_sync(0xffffffffu, lo2, m));
            hi2 = fmaxf(hi2, __shfl_xor_sync(0xffffffffu, hi2, m));
        }
        // exp(G_t - G_i) = row_t * col_i with the reference in the middle of the tile's range of
        // G; both factors stay within 2^+-126 when that range spans at most 250 powers of two,
        // otherwise the exponent is taken per entry.
        const float ref = 0.5f * (lo2 + hi2);
        float* tg = reinterpret_cast<float*>(sm + WY_TG) + buf * kTgFloats;
        tg[2 * lane] = g20; tg[2 * lane + 1] = g21;
        tg[64 + 2 * lane] = pb[0]; tg[64 + 2 * lane + 1] = pb[1];
        tg[128 + 2 * lane] = pb[0] * fast_exp2(g20 - ref); tg[128 + 2 * lane + 1] = pb[1] * fast_exp2(g21 - ref);
        tg[192 + 2 * lane] = fast_exp2(ref - g20); tg[192 + 2 * lane + 1] = fast_exp2(ref - g21);
        tg[256 + 2 * lane] = expf(GC - G0); tg[256 + 2 * lane + 1] = expf(GC - G1);
        if (lane == 0) reinterpret_cast<int*>(tg)[320] = (hi2 - lo2) <= 250.f;
    };

    // K K^T of the item-th item of this CTA into TMEM (warp 0; M = 128: rows 64..127 of A read the
    // 8 KB past the tile, their output is ignored)
    auto issue_kk = [&](int item) {
        const bool ok = __all_sync(0xffffffffu, item == 0 ? mbar_wait(&mb_k, 0, budget0)
                                                           : mbar_wait(&mb_k, item & 1, kWaitBudgetNs)) != 0;
        if (!ok) {
            if (lane == 0) { record_status(a.status, DELTAS_ERR_TIMEOUT, 21); s_fail = 1; }
            return;
        }
        tc_fence_after();
        const uint32_t id = idesc_bf16(128, 64, 0, 0);
#pragma unroll
        for (int s = 0; s < 8; ++s) {
            const uint64_t d = sdesc_sw128(smem_u32(sm + WY_K + (s >> 2) * 8192 + (s & 3) * 32), 16, 1024);
            mma_bf16(tm, d, d, id, s > 0);
        }
        mma_commit(&mb_kk);
        ++nkk;
    };

    const int first = (int)blockIdx.x;
    if (first < items) {
        if (tid == 0) load_k(first);
        if (warp == 7) {
            load_gb(first);
            tile_constants(first, 0);
            if (first + (int)gridDim.x < items) load_gb(first + (int)gridDim.x);
        }
    }
    __syncthreads();
    int c = 0;                                         // items done by this CTA (barrier phases)
    for (int it = first; it < items; it += (int)gridDim.x, ++c) {
        const float* tg = reinterpret_cast<const float*>(sm + WY_TG) + (c & 1) * kTgFloats;
        const float* sG2 = tg;                         // G * log2(e)
        const float* sBeta = tg + 64;
        const float* sRow = tg + 128;                  // beta_t 2^(G2_t - ref)
        const float* sCol = tg + 192;                  // 2^(ref - G2_i)
        const float* sDel = tg + 256;                  // exp(G_C - G_t)
        const int factored = reinterpret_cast<const int*>(tg)[320];
        if (warp == 0) issue_kk(c);
        const int q = warp & 3;
        if (q < 2 && warp != 4) {
            // TMEM lanes 0..63 hold K K^T: warps 0/4 rows 0..31, 1/5 rows 32..63; column half
            // (warp >> 2).  Warp 4's quarter (rows 0..31, cols 32..63) lies above the diagonal and
            // is never needed; warp 1's (rows 32..63, cols 0..31) is A21, stored split.
            const bool ok = mbar_wait_or_abort(&mb_kk, c & 1, kWaitBudgetNs, &s_fail);
            if (!ok && lane == 0) { record_status(a.status, DELTAS_ERR_TIMEOUT, 22); s_fail = 1; }
            tc_fence_after();
            const int t = 32 * q + lane, c0 = 32 * (warp >> 2);
            const uint32_t lane_off = (uint32_t)(32 * q) << 16;
            const float rt = factored ? sRow[t] : sBeta[t];
            const float G2t = sG2[t];
#pragma unroll
            for (int half = 0; half < 2; ++half) {     // 16 columns at a time
                const int cb = c0 + 16 * half;
                float kk[16], cf[16];
                tmem_ld16(tm + lane_off + cb, kk);
                const float* src = factored ? sCol : sG2;
#pragma unroll
                for (int e = 0; e < 4; ++e) {
                    const float4 v4 = *reinterpret_cast<const float4*>(src + cb + 4 * e);
                    cf[4 * e] = v4.x; cf[4 * e + 1] = v4.y; cf[4 * e + 2] = v4.z; cf[4 * e + 3] = v4.w;
                }
                tmem_ld_wait();
#pragma unroll
                for (int e = 0; e < 16; ++e) {
                    const float f = factored ? cf[e] : fast_exp2(G2t - cf[e]);
                    kk[e] = (cb + e < t) ? rt * f * kk[e] : 0.f;
                }
                if (half == 0 && lane >= 16 && (warp == 0 || warp == 5))   // A10 / A32, split
                    put_split16((warp == 0 ? sA10 : sA32) + (lane - 16) * kL1S, kk);
                if (warp == 1) {                       // A21, split
                    uint32_t* row = sA21 + (t - 32) * FA_S + 8 * half;
                    uint32_t h[8], l[8];
#pragma unroll
                    for (int i = 0; i < 8; ++i) split2(kk[2 * i], kk[2 * i + 1], h[i], l[i]);
                    *reinterpret_cast<uint4*>(row) = make_uint4(h[0], h[1], h[2], h[3]);
                    *reinterpret_cast<uint4*>(row + 4) = make_uint4(h[4], h[5], h[6], h[7]);
                    *reinterpret_cast<uint4*>(row + 16) = make_uint4(l[0], l[1], l[2], l[3]);
                    *reinterpret_cast<uint4*>(row + 20) = make_uint4(l[4], l[5], l[6], l[7]);
                } else {
#pragma unroll
                    for (int e = 0; e < 4; ++e)
                        *reinterpret_cast<float4*>(fA + t * FA_S + cb + 4 * e) =
                            make_float4(kk[4 * e], kk[4 * e + 1], kk[4 * e + 2], kk[4 * e + 3]);
                }
            }
        }
        tc_fence_before();
        __syncthreads();
        if (s_fail) break;
        const int nxt = it + (int)gridDim.x;
        // level 0: four 16 x 16 diagonal blocks of (I + A)^-1, one column per thread (warps 0-1);
        // meanwhile warp 7 prepares the next item's constants and loads the one after
        if (tid < 64) {
            const int B = tid >> 4, jc = tid & 15, o = 16 * B;
            float x[16];
#pragma unroll
            for (int rr = 0; rr < 16; ++rr) x[rr] = (rr == jc) ? 1.f : 0.f;
#pragma unroll
            for (int rr = 1; rr < 16; ++rr) {
                float s0 = 0.f, s1 = 0.f;              // two chains: half the dependent FMAs
#pragma unroll
                for (int cc = 0; cc < rr; cc += 4) {
                    const float4 av = *reinterpret_cast<const float4*>(fA + (o + rr) * FA_S + o + cc);
                    s0 = fmaf(av.x, x[cc], s0);
                    if (cc + 1 < rr) s1 = fmaf(av.y, x[cc + 1], s1);
                    if (cc + 2 < rr) s0 = fmaf(av.z, x[cc + 2], s0);
                    if (cc + 3 < rr) s1 = fmaf(av.w, x[cc + 3], s1);
                }
                if (rr > jc) x[rr] = -(s0 + s1);
            }
#pragma unroll
            for (int rr = 0; rr < 16; ++rr) fX[(o + rr) * FX_S + o + jc] = x[rr];
            if (B == 1) {                              // X11' row-major
#pragma unroll
                for (int rr = 0; rr < 16; ++rr) put_split(sX11r + rr * kL1S, jc, x[rr], 8);
            } else if (B == 2) {                       // X22' n-major
                put_split16(sX22n + jc * kL1S, x);
            }
            if (B < 2) {                               // X11, n-major: row o + jc holds column o + jc
                uint32_t* row = sX11 + (o + jc) * FA_S;
                if (B == 1) {                          // X[0..16][16..32] = 0 (the K tile overwrote it)
                    const uint4 z = make_uint4(0u, 0u, 0u, 0u);
                    *reinterpret_cast<uint4*>(row) = z; *reinterpret_cast<uint4*>(row + 4) = z;
                    *reinterpret_cast<uint4*>(row + 16) = z; *reinterpret_cast<uint4*>(row + 20) = z;
                }
#pragma unroll
                for (int e = 0; e < 2; ++e) {
                    uint32_t h[4], l[4];
#pragma unroll
                    for (int i = 0; i < 4; ++i) split2(x[8 * e + 2 * i], x[8 * e + 2 * i + 1], h[i], l[i]);
                    *reinterpret_cast<uint4*>(row + o / 2 + 4 * e) = make_uint4(h[0], h[1], h[2], h[3]);
                    *reinterpret_cast<uint4*>(row + 16 + o / 2 + 4 * e) = make_uint4(l[0], l[1], l[2], l[3]);
                }
            } else {                                   // X22, row-major
#pragma unroll
                for (int rr = 0; rr < 16; ++rr) put_split(sX22 + (o - 32 + rr) * FX_S, o - 32 + jc, x[rr]);
            }
        } else if (warp == 7 && nxt < items) {
            tile_constants(nxt, (c + 1) & 1);
            if (nxt + (int)gridDim.x < items) load_gb(nxt + (int)gridDim.x);
        }
        __syncthreads();
        // level 1: X[2p+1][2p] = -X[2p+1][2p+1] (A[2p+1][2p] X[2p][2p]) for the 16 x 16 blocks,
        // p = 0, 1; warps 0-3 take (p, 8-column half) = (warp / 2, warp % 2)
        const int g = lane >> 2, tq = lane & 3;
        if (warp < 4) {
            const int p = warp >> 1, nc = 8 * (warp & 1);
            float d[4] = {0.f, 0.f, 0.f, 0.f};
            if (p == 0) mma_split_bf16<1>(d, sA10, kL1S, 8, 0, sX11, FA_S, 16, nc, lane);    // A10 X00
            else        mma_split_bf16<1>(d, sA32, kL1S, 8, 0, sX22n, kL1S, 8, nc, lane);   // A32 X22'
            uint32_t* P = sP1 + p * 16 * kL1S;         // n-major
            put_split(P + (nc + 2 * tq) * kL1S, g, d[0], 8);
            put_split(P + (nc + 2 * tq + 1) * kL1S, g, d[1], 8);
            put_split(P + (nc + 2 * tq) * kL1S, g + 8, d[2], 8);
            put_split(P + (nc + 2 * tq + 1) * kL1S, g + 8, d[3], 8);
        }
        __syncthreads();
        if (warp < 4) {
            const int p = warp >> 1, nc = 8 * (warp & 1);
            const int ro = 16 * (2 * p + 1), co = 16 * (2 * p);
            const uint32_t* P = sP1 + p * 16 * kL1S;
            float d[4] = {0.f, 0.f, 0.f, 0.f};
            if (p == 0) mma_split_bf16<1>(d, sX11r, kL1S, 8, 0, P, kL1S, 8, nc, lane);        // X11' P1
            else        mma_split_bf16<1>(d, sX22 + 16 * FX_S + 8, FX_S, 16, 0, P, kL1S, 8, nc, lane);  // X33' P1'
            fX[(ro + g) * FX_S + co + nc + 2 * tq] = -d[0]; fX[(ro + g) * FX_S + co + nc + 2 * tq + 1] = -d[1];
            fX[(ro + g + 8) * FX_S + co + nc + 2 * tq] = -d[2]; fX[(ro + g + 8) * FX_S + co + nc + 2 * tq + 1] = -d[3];
            if (p == 0) {                              // X[16..32][0..16] into X11, n-major
                put_split(sX11 + (nc + 2 * tq) * FA_S, 16 + g, -d[0]);
                put_split(sX11 + (nc + 2 * tq + 1) * FA_S, 16 + g, -d[1]);
                put_split(sX11 + (nc + 2 * tq) * FA_S, 24 + g, -d[2]);
                put_split(sX11 + (nc + 2 * tq + 1) * FA_S, 24 + g, -d[3]);
            } else {                                   // X[48..64][32..48] into X22, row-major
                put_split(sX22 + (16 + g) * FX_S, nc + 2 * tq, -d[0]);
                put_split(sX22 + (16 + g) * FX_S, nc + 2 * tq + 1, -d[1]);
                put_split(sX22 + (24 + g) * FX_S, nc + 2 * tq, -d[2]);
                put_split(sX22 + (24 + g) * FX_S, nc + 2 * tq + 1, -d[3]);
            }
        }
        __syncthreads();
        // level 2: X[32:64][0:32] = -X[32:64][32:64] (A[32:64][0:32] X[0:32][0:32]) from the split
        // operands; warp w takes the 16 x 8 output tile (w / 4, w % 4).  P = A21 X11 goes to fT
        // split and n-major.
        {
            const int mr = 16 * (warp >> 2), nc = 8 * (warp & 3);
            float d[4] = {0.f, 0.f, 0.f, 0.f};
            mma_split_bf16<2>(d, sA21, FA_S, 16, mr, sX11, FA_S, 16, nc, lane);
            put_split(sP + (nc + 2 * tq) * kPS, mr + g, d[0]);
            put_split(sP + (nc + 2 * tq + 1) * kPS, mr + g, d[1]);
            put_split(sP + (nc + 2 * tq) * kPS, mr + g + 8, d[2]);
            put_split(sP + (nc + 2 * tq + 1) * kPS, mr + g + 8, d[3]);
        }
        __syncthreads();
        // A (fp32 and split) has been read for the last time: the next item's K tile lands there
        if (tid == 0 && nxt < items) load_k(nxt);
        {
            const int mr = 16 * (warp >> 2), nc = 8 * (warp & 3);
            float d[4] = {0.f, 0.f, 0.f, 0.f};
            mma_split_bf16<2>(d, sX22, FX_S, 16, mr, sP, kPS, 16, nc, lane);
            fX[(32 + mr + g) * FX_S + nc + 2 * tq] = -d[0]; fX[(32 + mr + g) * FX_S + nc + 2 * tq + 1] = -d[1];
            fX[(32 + mr + g + 8) * FX_S + nc + 2 * tq] = -d[2]; fX[(32 + mr + g + 8) * FX_S + nc + 2 * tq + 1] = -d[3];
        }
        __syncthreads();
        // T~ = diag(exp(G_C - G)) X diag(beta) (upper part zero), split into the record's (hi, lo)
        // images; for the read-out T = X diag(beta)
        {
            uint8_t* rec = a.rec + (size_t)rec_of(it) * rec_bytes(a.out);
#pragma unroll
            for (int m = 0; m < 2; ++m) {
                const int e = tid + kWyThreads * m;
                const int t = e >> 3, c8 = e & 7;
                uint4 vh = make_uint4(0u, 0u, 0u, 0u), vl = vh;
                if (8 * c8 <= t) {                     // chunks right of the diagonal stay zero
                    const float dt = a.out ? 1.f : sDel[t];
                    const float4 x0 = *reinterpret_cast<const float4*>(fX + t * FX_S + 8 * c8);
                    const float4 x1 = *reinterpret_cast<const float4*>(fX + t * FX_S + 8 * c8 + 4);
                    const float4 b0 = *reinterpret_cast<const float4*>(sBeta + 8 * c8);
                    const float4 b1 = *reinterpret_cast<const float4*>(sBeta + 8 * c8 + 4);
                    const float xs[8] = {x0.x * b0.x, x0.y * b0.y, x0.z * b0.z, x0.w * b0.w,
                                         x1.x * b1.x, x1.y * b1.y, x1.z * b1.z, x1.w * b1.w};
                    float x[8];
#pragma unroll
                    for (int k = 0; k < 8; ++k) x[k] = (8 * c8 + k <= t) ? dt * xs[k] : 0.f;
                    split8(x, vh, vl);
                }
                *reinterpret_cast<uint4*>(rec + sw128_offset(t, c8)) = vh;
                *reinterpret_cast<uint4*>(rec + 8192 + sw128_offset(t, c8)) = vl;
            }
        }
        // the next item's level 0 rewrites fX's diagonal blocks: everyone has read this one's
        __syncthreads();
    }
    if (tid == 0 && s_fail) {
        // after a failure: the last K load and K K^T product issued land before TMEM is freed
        if (nk > 0) mbar_wait(&mb_k, (nk - 1) & 1, kWaitBudgetNs);
        if (nkk > 0) mbar_wait(&mb_kk, (nkk - 1) & 1, kWaitBudgetNs);
    }
    tc_fence_before();
    __syncthreads();
    if (warp == 0) {
        tc_fence_after();
        tmem_dealloc(tm, kWyTmemCols);
    }
}

// =============================================================================================
// Update kernel: the state chain
// =============================================================================================
__device__ __forceinline__ int ho_load_acquire(const int32_t* p) {
    int v;
    asm volatile("ld.acquire.gpu.global.b32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
    return v;
}
__device__ __forceinline__ void ho_store_release(int32_t* p, int v) {
    asm volatile("st.release.gpu.global.b32 [%0], %1;" :: "l"(p), "r"(v) : "memory");
}
// orders the tensor copies' global accesses with the generic ones around a hand-over flag
__device__ __forceinline__ void fence_proxy_async_global() {
    asm volatile("fence.proxy.async.global;" ::: "memory");
}

constexpr int kChainWarps = 16;
constexpr int kChain = 32 * kChainWarps;         // chain threads
constexpr int kMmaWarp = kChainWarps;            // 16
constexpr int kLoadWarp = kChainWarps + 1;       // 17
constexpr int kStateWarp = kChainWarps + 2;      // 18
constexpr int kThreads = kChain + 96;
constexpr uint32_t kTmemCols = 512;
constexpr uint32_t TM_S = 0, TM_SB = 128, TM_X = 256, TM_U = 320, TM_V = 384;

// shared-memory map (bytes from a 1024-aligned base)
constexpr uint32_t SM_K = 0;                     // 3 x 16 KB: K tile, 2 column blocks (d 0-63, 64-127) x 64 rows x 128 B
constexpr uint32_t SM_K32 = 49152;               // 32 KB: K in fp32 (the B operand of X), 4 column blocks
                                                 // (32 dims) x 64 rows x 128 B, SW128
constexpr uint32_t SM_V = 81920;                 // 2 x 16 KB: V tile (tile parity), layout of K
constexpr uint32_t SM_R = 114688;                // 2 x kRecSlot: WY records (tile parity)
constexpr uint32_t kRecSlot = 17408;             // 1024-aligned slots
constexpr uint32_t SM_I = SM_R + 2 * kRecSlot;   // 8 KB: 64 x 64 bfloat16 identity, K-major SW128
constexpr uint32_t SM_SB = SM_I + 8192;          // 64 KB: state staging, 4 column blocks x 128 rows x 128 B, SW128
constexpr uint32_t SM_BYTES = SM_SB + 65536;
constexpr uint32_t kSmemAlloc = SM_BYTES + 1024;
static_assert(SM_I % 1024 == 0 && SM_SB % 1024 == 0 && kRecSlot >= kRecBytesOut, "shared-memory map");
static_assert(SM_SB >= 131072, "the segment combine's images ([0, 128 KB)) lie below the staging buffer");
static_assert(kSmemAlloc <= 232448, "shared memory budget");

// The staging buffer holds a head's [d_v][d_k] fp32 state as four column blocks of 32 floats, each
// 128 rows x 128 bytes with the 128-byte swizzle (16-byte chunk ^ (row & 7)) that TMA writes and
// reads; eight threads reading chunk c of eight consecutive rows (one row per thread) hit distinct
// banks.  Float offset of 16-byte chunk `chunk` (0..31) of row `row`:
__device__ __forceinline__ int sb_idx(int row, int chunk) {
    return (chunk >> 3) * 4096 + row * 32 + (((chunk & 7) ^ (row & 7)) << 2);
}

struct TcArgs {
    int L, Hk, Hv, T, n_tiles;
    float* state;
    float* partials;
    float* wnorm;
    const uint8_t* rec;
    int32_t* status;
    int split;               // run equal tile runs (ChainSched), when the host found it faster
    // hand-over between neighbouring CTAs of a head split between them (see ChainSched): one
    // entry per CTA boundary i (CTA i -> CTA i + 1)
    int32_t* ho_flag;        // [grid] the state after the first part is in the hand-over map
    int32_t* ho_wflag;       // [grid] the first part's write-size sum is in ho_wsum
    float* ho_wsum;          // [grid]
    // segments (see ChainSched): seg = 2 runs each head's tiles as two segments on three CTAs
    int seg;
    uint8_t* ho_base;        // the hand-over states (the hmap rows): CTA i's 64 KB at ho_base + 64 KB i
    // read-out: each token's write u_t, and the state at the start of every 128-token block,
    // both as B operands of the read-out's MMAs (N = d_v rows, K-major, no swizzle): chunks of 4
    // consecutive K values, each chunk's 128 rows of 16 bytes contiguous (a warp's 32 rows of one
    // chunk are one 512-byte store)
    float* ubuf;             // [L * Hv][16 n_tiles token chunks][d_v][4] fp32
    float* snap;             // [L * Hv][n_blk][32 d_k chunks][d_v][4] fp32
    int n_blk;               // ceil(n_tiles / 2)
};

// The CTA's work: a sequence of slots, each a run of consecutive tiles of one head.  By default
// the CTA owns heads blockIdx.x, blockIdx.x + gridDim.x, ... whole.  When the heads do not divide
// evenly among the CTAs and the host estimates it faster (a.split), the CTAs instead take equal
// runs of the tile sequence in head order, so that the slowest CTA has one tile more than the
// fastest instead of a whole head more; a head cut by a run boundary is shared by two neighbours.  CTA i runs the head
// it shares with CTA i + 1 first (its first tiles; the state at the cut goes to hand-over entry i)
// and the head it shares with CTA i - 1 last (its last tiles, from hand-over entry i - 1), so the
// second part of a shared head is never waited for before its first part is long finished.
//
// Segments.  When the heads are few (a single layer: 32 heads on 152 SMs) the tiles of one head
// run in series on one CTA while most SMs idle.  A run of tiles is an affine map of the state,
// S_end = S_start A + B, so the host may cut each head's tiles in two halves on three CTAs: CTA 0
// runs the first half from the state, CTA 1 the second half from S = I with v = 0 (its end state
// is A, written as the bfloat16 (hi, lo) images of an MN-major MMA operand) and CTA 2 from S = 0
// (B, fp32); both raise their hand-over flag.  CTA 0 then waits for them (bounded), forms
// S_0 A by three tcgen05 products from its own state and A's images, sets S~ = S_0 A + B (B through
// its staging buffer) and leaves through the ordinary head boundary (S_after, drift partials).
struct ChainSched {
    int seg_mode;              // 0: not segmented; 1: segment 0 (from the state); 2: from I, v = 0;
                               // 3: from 0
    int seg_lh, seg_tb, seg_te;
    int split;
    int pre_lh, pre_len;       // first slot: tiles [0, pre_len) of head pre_lh (none if pre_len == 0)
    int full0, n_full;         // then n_full whole heads from full0 (every gridDim.x-th if !split)
    int suf_lh, suf_from;      // last slot: tiles [suf_from, n) of head suf_lh (none if suf_from == 0)
    int n_slots, NJ;
    __device__ __forceinline__ void init(const TcArgs& a, bool segmented) {
        const int n = a.n_tiles, G = (int)gridDim.x, i = (int)blockIdx.x, H = a.L * a.Hv;
        seg_mode = 0;
        if (segmented) {
            const int per = 2 * a.seg - 1, hd = i / per, r = i - hd * per, sg = (r + 1) >> 1;
            seg_mode = r == 0 ? 1 : (r & 1) ? 2 : 3;
            seg_lh = hd;
            seg_tb = (int)((long long)sg * n / a.seg);          // balanced cuts: >= 4 tiles each
            seg_te = (int)((long long)(sg + 1) * n / a.seg);
            split = 0;
            pre_lh = suf_lh = -1; pre_len = suf_from = 0;
            full0 = hd; n_full = n_slots = 1; NJ = seg_te - seg_tb;
            return;
        }
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
        if (seg_mode) { lh = seg_lh; tb = seg_tb; te = seg_te; return; }
        tb = 0; te = n;
        if (!split) { lh = full0 + k * (int)gridDim.x; return; }
        if (is_prefix(k)) { lh = pre_lh; te = pre_len; return; }
        if (is_suffix(k)) { lh = suf_lh; tb = suf_from; return; }
        lh = full0 + k - (pre_len > 0 ? 1 : 0);
    }
};

// Where the CTA's current tile lies: slot k, tile jt (of [tb, te)) of head lh = (layer l, value
// head h), key head kh.  Each role walks the tiles in order; a step costs integer divisions only
// when it crosses into the next slot.
struct TileCursor {
    int k, jt, te, lh, l, h, kh;
    __device__ __forceinline__ void set_slot(int slot, const ChainSched& sc, const TcArgs& a) {
        int tb;
        k = slot;
        sc.slot(slot, a.n_tiles, lh, tb, te);
        jt = tb;
        l = lh / a.Hv; h = lh - l * a.Hv;
        kh = (int)(((long long)h * a.Hk) / a.Hv);
    }
    __device__ __forceinline__ void init(const ChainSched& sc, const TcArgs& a) {
        if (sc.n_slots > 0) set_slot(0, sc, a);
    }
    __device__ __forceinline__ void next(const ChainSched& sc, const TcArgs& a) {
        if (++jt == te && k + 1 < sc.n_slots) set_slot(k + 1, sc, a);
    }
};

template <bool kOut, bool kSeg>
__global__ void __launch_bounds__(kThreads, 1)
gdn_update_tc_kernel(const __grid_constant__ CUtensorMap kmap, const __grid_constant__ CUtensorMap vmap,
                     const __grid_constant__ CUtensorMap smap, const __grid_constant__ CUtensorMap hmap,
                     TcArgs a)
{
    extern __shared__ uint8_t smem_raw[];
    uint8_t* sm = smem_raw + ((1024 - (smem_u32(smem_raw) & 1023)) & 1023);
    // copies -> roles: K (3), V (2), WY records (2) full; MMA -> loader: their empties; state
    // staging full (mb_st) and released by the chain (mb_sfree); MMA -> chain: x, u, s; chain ->
    // MMA: ready flags.
    __shared__ uint64_t mb_tk[3], mb_ke[3], mb_tv[2], mb_ve[2], mb_tr[2], mb_re[2];
    __shared__ uint64_t mb_st, mb_sfree, mb_x, mb_u, mb_s, mb_sready, mb_xready, mb_uready, mb_fin;
    __shared__ uint64_t mb_end, mb_cimg, mb_cd, mb_ca;   // segment combine (CTA 0 of a head): MMAs done,
                                                         // S_0 images, the product, A's images
    __shared__ uint32_t s_tmem;
    __shared__ int s_abort;
    __shared__ float s_red[2][kChainWarps];
    __shared__ float s_u2[2][kC];                 // per-token squared write sizes (tile parity)
    volatile int* abort_flag = &s_abort;

    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int n = a.n_tiles;
    // Persistent CTA: its slots (ChainSched) form one sequence of NJ tiles, over which every role
    // keeps its barrier phases.
    ChainSched sch;
    sch.init(a, kSeg);
    const int n_slots = sch.n_slots;
    const int NJ = sch.NJ;

    if (warp == kMmaWarp) {
        tmem_alloc(&s_tmem, kTmemCols);
        tmem_relinquish();
        if (lane == 0) {
            for (int b = 0; b < 3; ++b) { mbar_init(&mb_tk[b], 1); mbar_init(&mb_ke[b], 1); }
            for (int b = 0; b < 2; ++b) {
                mbar_init(&mb_tv[b], 1); mbar_init(&mb_ve[b], 1);
                mbar_init(&mb_tr[b], 1); mbar_init(&mb_re[b], 1);
            }
            mbar_init(&mb_st, 1); mbar_init(&mb_sfree, kChainWarps);
            mbar_init(&mb_x, 1); mbar_init(&mb_u, 1); mbar_init(&mb_s, 1);
            mbar_init(&mb_sready, kChainWarps); mbar_init(&mb_xready, kChainWarps);
            mbar_init(&mb_uready, kChainWarps);
            mbar_init(&mb_fin, 1);
            mbar_init(&mb_end, 1); mbar_init(&mb_cimg, kChainWarps); mbar_init(&mb_cd, 1); mbar_init(&mb_ca, 1);
            fence_barrier_init();
        }
    }
    if (warp == kLoadWarp && lane == 0) { prefetch_tensormap(&kmap); prefetch_tensormap(&vmap); }
    if (warp == kStateWarp && lane == 0) { prefetch_tensormap(&smap); prefetch_tensormap(&hmap); }
    if (tid < kChain) {
        // the 64 x 64 identity (B operand of V^T I): row t holds 1.0 at column t
        const int t = tid >> 3, c8 = tid & 7;
        uint32_t w[4] = {0u, 0u, 0u, 0u};
        if ((t >> 3) == c8) w[(t & 7) >> 1] = (t & 1) ? 0x3F800000u : 0x00003F80u;
        *reinterpret_cast<uint4*>(sm + SM_I + sw128_offset(t, c8)) = make_uint4(w[0], w[1], w[2], w[3]);
        fence_async_smem();
    }
    if (tid == 0) s_abort = 0;
    if (tid < 2 * kC) s_u2[tid >> 6][tid & (kC - 1)] = 0.f;
    grid_dep_launch();                                 // the next kernel (the score) may be scheduled
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tm = s_tmem;

    if (warp == kMmaWarp) {
        // =========================================================== MMA issue (converged warp;
        // one elected lane issues each group and commits it)
        const uint64_t dK = sdesc_sw128(smem_u32(sm + SM_K), 8192, 1024);    // MN-major B of MMA_S
        const uint64_t dK32 = sdesc_sw128(smem_u32(sm + SM_K32), 16, 1024);
        const uint64_t dV = sdesc_sw128(smem_u32(sm + SM_V), 8192, 1024);    // MN-major A of V^T I
        const uint64_t dR = sdesc_sw128(smem_u32(sm + SM_R), 16, 1024);
        const uint64_t dI = sdesc_sw128(smem_u32(sm + SM_I), 16, 1024);
        // Each group's operands are formed before the wait that releases it, so that only the
        // MMA instructions themselves follow the wait (this warp shares its scheduler with four
        // chain warps).
        // V region <- V(J)^T: A = the V tile read MN-major (k-step s = tokens 16 s ..), B = I.  V(J)'s
        // buffer is released when the product completes.
        auto issue_vi = [&](int J, uint64_t budget) -> bool {
            uint64_t av[4], bv[4];
#pragma unroll
            for (int s = 0; s < 4; ++s) {
                av[s] = dadd(dV, (J & 1) * 16384 + s * 2048); bv[s] = dadd(dI, s * 32);
                pin(av[s]); pin(bv[s]);
            }
            if (!warp_wait(&mb_tv[J & 1], (J >> 1) & 1, budget, abort_flag)) return false;
            tc_fence_after();
            if (elect_one()) mma4_bf16_ss_1t(tm + TM_V, av, bv, idesc_bf16(128, 64, 1, 0), 0);
            __syncwarp();
            mma_commit(&mb_ve[J & 1]);
            return true;
        };
        // the workspace's wait budget bounds this first wait (V of the CTA's first tile); the
        // per-tile waits keep the fixed bound (a bound read at run time in every wait of this
        // latency-bound chain measured 5 % slower)
        bool ok = NJ == 0 || issue_vi(0, wait_budget_ns(a.status));
        if (!ok) fail(a.status, abort_flag, 1);
        for (int j = 0; ok && j < NJ; ++j) {           // j: global tile index
            {   // X region <- S~ K^T: A = the fp32 state from TMEM read as tf32 (8 columns per K = 8
                // step), B = K in fp32.  Tile j ready for X: K(j) is converted and, at a head's first
                // tile, the state is in TMEM (otherwise MMA_S(j-1), issued before, produces it in pipe
                // order).
                uint32_t ax[4][4];
                uint64_t bx[4][4];
#pragma unroll
                for (int s = 0; s < 16; ++s) {
                    ax[s >> 2][s & 3] = tm + TM_S + 8 * s;
                    bx[s >> 2][s & 3] = dadd(dK32, (s >> 2) * 8192 + (s & 3) * 32);
                    pin(ax[s >> 2][s & 3]); pin(bx[s >> 2][s & 3]);
                }
                if (!warp_wait(&mb_sready, j & 1, kWaitBudgetNs, abort_flag)) { fail(a.status, abort_flag, 2); break; }
                tc_fence_after();
                if (elect_one()) {
#pragma unroll
                    for (int g4 = 0; g4 < 4; ++g4) mma4_tf32_ta_1t(tm + TM_X, ax[g4], bx[g4], idesc_tf32(128, 64), g4 != 0);
                }
                __syncwarp();
                mma_commit(&mb_x);
            }
            {   // U region <- W^T T~^T with W (hi, lo) packed in place in X (k-step s: hi at column
                // 16 s, lo at 16 s + 8): W hi T~ hi + W hi T~ lo + W lo T~ hi
                uint32_t au[3][4];
                uint64_t bu[3][4];
                const uint32_t rb = (j & 1) * kRecSlot;
#pragma unroll
                for (int part = 0; part < 3; ++part) {
#pragma unroll
                    for (int s = 0; s < 4; ++s) {
                        au[part][s] = tm + TM_X + 16 * s + (part == 2 ? 8 : 0);
                        bu[part][s] = dadd(dR, rb + (part == 1 ? 8192 : 0) + s * 32);
                        pin(au[part][s]); pin(bu[part][s]);
                    }
                }
                if (!warp_wait(&mb_xready, j & 1, kWaitBudgetNs, abort_flag)) { fail(a.status, abort_flag, 5); break; }
                if (!warp_wait(&mb_tr[j & 1], (j >> 1) & 1, kWaitBudgetNs, abort_flag)) { fail(a.status, abort_flag, 3); break; }
                tc_fence_after();
                if (elect_one()) {
#pragma unroll
                    for (int part = 0; part < 3; ++part)
                        mma4_bf16_ta_1t(tm + TM_U, au[part], bu[part], idesc_bf16(128, 64, 0, 0), part != 0);
                }
                __syncwarp();
                mma_commit(&mb_u);
                mma_commit(&mb_re[j & 1]);             // record slot free once MMA_U(j) has read T~
            }
            // the next tile's V^T into the V region (its last reader, the W pass of tile j, has
            // finished: MMA_U(j) waited for xready)
            if (j + 1 < NJ && !issue_vi(j + 1, kWaitBudgetNs)) { fail(a.status, abort_flag, 4); break; }
            {   // S~ += U~^T K  (A: U~ hi / lo packed in place in U; K read MN-major)
                uint32_t as_[2][4];
                uint64_t bs[2][4];
                const uint32_t kb = (j % 3) * 16384;
#pragma unroll
                for (int part = 0; part < 2; ++part) {
#pragma unroll
                    for (int s = 0; s < 4; ++s) {
                        as_[part][s] = tm + TM_U + 16 * s + (part == 1 ? 8 : 0);
                        bs[part][s] = dadd(dK, kb + s * 2048);
                        pin(as_[part][s]); pin(bs[part][s]);
                    }
                }
                if (!warp_wait(&mb_uready, j & 1, kWaitBudgetNs, abort_flag)) { fail(a.status, abort_flag, 7); break; }
                tc_fence_after();
                if (elect_one()) {
#pragma unroll
                    for (int part = 0; part < 2; ++part)
                        mma4_bf16_ta_1t(tm + TM_S, as_[part], bs[part], idesc_bf16(128, 128, 0, 1), 1);
                }
                __syncwarp();
                mma_commit(&mb_s);
                mma_commit(&mb_ke[j % 3]);             // K(j)'s buffer free once MMA_S(j) has read it
            }
        }
        if (kSeg && sch.seg_mode == 1 && ok) {
            // segment combine: S_0 A into the X / U columns, from CTA 0's state images (K-major) and
            // A's images (MN-major), once every MMA of the chain has completed
            mma_commit(&mb_end);
            if (warp_wait(&mb_cimg, 0, kWaitBudgetNs, abort_flag) && warp_wait(&mb_ca, 0, kWaitBudgetNs, abort_flag)) {
                tc_fence_after();
                if (elect_one()) {
                    const uint32_t id = idesc_bf16(128, 128, 0, 1);
#pragma unroll
                    for (int term = 0; term < 3; ++term) {   // S0_hi A_hi, S0_hi A_lo, S0_lo A_hi
                        const uint32_t xb = term == 2 ? 32768u : 0u, ab = term == 1 ? 98304u : 65536u;
#pragma unroll
                        for (int s = 0; s < 8; ++s) {        // K = 16 per MMA
                            const uint64_t da = sdesc_sw128(smem_u32(sm + xb + (s >> 2) * 16384 + (s & 3) * 32), 16, 1024);
                            const uint64_t db = sdesc_sw128(smem_u32(sm + ab + s * 2048), 16384, 1024);
                            mma_bf16_1t(tm + TM_X, da, db, id, (term | s) != 0);
                        }
                    }
                }
                __syncwarp();
                mma_commit(&mb_cd);
            } else {
                fail(a.status, abort_flag, 8);
            }
        }
        if (__any_sync(0xffffffffu, *abort_flag != 0)) {
            mma_commit(&mb_fin);                       // every MMA this warp issued has completed
            mbar_wait(&mb_fin, 0, kWaitBudgetNs);
        }
        __syncwarp();
    } else if (warp == kLoadWarp) {
        // =========================================================== K, V, records in tile order,
        // each into its buffer once the MMA that last read the buffer has completed
        TileCursor cc;
        cc.init(sch, a);
        int kp[3] = {-1, -1, -1}, vp[2] = {-1, -1}, rp[2] = {-1, -1};   // last tile loaded per buffer
        // the kernel may start while the factor kernel finishes (its set-up and the first state
        // load overlap that tail); the records it wrote are read only after it has completed
        grid_dep_wait();
        for (int J = 0; J < NJ; ++J) {
            const int bk = J % 3, b2 = J & 1;
            if (J >= 3 && !warp_wait(&mb_ke[bk], ((J / 3) - 1) & 1, kWaitBudgetNs, abort_flag)) { fail(a.status, abort_flag, 30); break; }
            if (elect_one()) {
                uint8_t* dst = sm + SM_K + bk * 16384;
                mbar_arrive_expect_tx(&mb_tk[bk], 16384);
                tma_load_4d(dst, &kmap, &mb_tk[bk], 0, cc.kh, cc.jt * kC, cc.l);
                tma_load_4d(dst + 8192, &kmap, &mb_tk[bk], 64, cc.kh, cc.jt * kC, cc.l);
            }
            __syncwarp();
            kp[bk] = J;
            if (J >= 2 && !warp_wait(&mb_ve[b2], ((J >> 1) - 1) & 1, kWaitBudgetNs, abort_flag)) { fail(a.status, abort_flag, 31); break; }
            if (elect_one()) {
                uint8_t* dst = sm + SM_V + b2 * 16384;
                mbar_arrive_expect_tx(&mb_tv[b2], 16384);
                tma_load_4d(dst, &vmap, &mb_tv[b2], 0, cc.h, cc.jt * kC, cc.l);
                tma_load_4d(dst + 8192, &vmap, &mb_tv[b2], 64, cc.h, cc.jt * kC, cc.l);
            }
            __syncwarp();
            vp[b2] = J;
            if (J >= 2 && !warp_wait(&mb_re[b2], ((J >> 1) - 1) & 1, kWaitBudgetNs, abort_flag)) { fail(a.status, abort_flag, 32); break; }
            if (elect_one()) {
                constexpr uint32_t RB = rec_bytes(kOut);
                mbar_arrive_expect_tx(&mb_tr[b2], RB);
                bulk_load_tx(sm + SM_R + b2 * kRecSlot, a.rec + ((size_t)cc.lh * n + cc.jt) * RB, RB, &mb_tr[b2]);
            }
            __syncwarp();
            rp[b2] = J;
            cc.next(sch, a);
        }
        if (__any_sync(0xffffffffu, *abort_flag != 0) && lane == 0) {
            // every copy this warp issued lands before the CTA ends
            for (int b = 0; b < 3; ++b)
                if (kp[b] >= 0) mbar_wait(&mb_tk[b], (kp[b] / 3) & 1, kWaitBudgetNs);
            for (int b = 0; b < 2; ++b) {
                if (vp[b] >= 0) mbar_wait(&mb_tv[b], (vp[b] >> 1) & 1, kWaitBudgetNs);
                if (rp[b] >= 0) mbar_wait(&mb_tr[b], (rp[b] >> 1) & 1, kWaitBudgetNs);
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
        // i - 1, once that entry's flag is set (bounded wait).
        if (lane == 0 && n_slots > 0) {
            float* sbuf = reinterpret_cast<float*>(sm + SM_SB);
            const int me = (int)blockIdx.x;
            int loads = 0, seen = 0;                   // copies into the staging buffer issued / landed
            auto load_rows = [&](const CUtensorMap* map, int row) {
                mbar_arrive_expect_tx(&mb_st, kD * kD * 4);
#pragma unroll
                for (int b = 0; b < 4; ++b) tma_load_2d(sbuf + 4096 * b, map, &mb_st, 32 * b, row);
                ++loads;
            };
            auto load_state = [&](int slot) -> bool {
                int lh, tb, te;
                sch.slot(slot, n, lh, tb, te);
                if (kSeg && sch.seg_mode >= 2) { mbar_arrive(&mb_st); return true; }   // the chain forms it
                if (!sch.is_suffix(slot)) { load_rows(&smap, lh * kD); return true; }
                grid_dep_wait();                       // the factor kernel reset the flags
                const uint64_t t0 = global_ns();
                while (ho_load_acquire(a.ho_flag + me - 1) == 0) {
                    if (*abort_flag || global_ns() - t0 > kWaitBudgetNs) return false;
                    __nanosleep(64);
                }
                fence_proxy_async_global();
                load_rows(&hmap, (me - 1) * kD);
                return true;
            };
            int ca = 0;                                // (segment combine) A's images copy issued
            auto wait_flag = [&](int idx) -> bool {    // hand-over entry idx published (bounded)
                grid_dep_wait();                       // (the factor kernel reset the flags)
                const uint64_t t0 = global_ns();
                while (ho_load_acquire(a.ho_flag + idx) == 0) {
                    if (*abort_flag || global_ns() - t0 > kWaitBudgetNs) return false;
                    __nanosleep(64);
                }
                fence_proxy_async_global();
                return true;
            };
            auto final_phase = [&]() -> bool {         // what the boundary after the last slot reads
                if (sch.is_suffix(n_slots - 1)) { load_rows(&smap, sch.suf_lh * kD); return true; }
                if (kSeg && sch.seg_mode == 1) {
                    // segment combine: B (CTA me + 2) into the staging buffer; A's images (CTA me + 1)
                    // into the tile buffers once every MMA of the chain has completed
                    if (!wait_flag(me + 2)) return false;
                    load_rows(&hmap, (me + 2) * kD);
                    if (!mbar_wait_or_abort(&mb_end, 0, kWaitBudgetNs, abort_flag) || !wait_flag(me + 1)) return false;
                    mbar_arrive_expect_tx(&mb_ca, 65536);
                    bulk_load_tx(sm + 65536, a.ho_base + (size_t)(me + 1) * 65536, 65536, &mb_ca);
                    ca = 1;
                    return true;
                }
                mbar_arrive(&mb_st);
                return true;
            };
            bool ok = load_state(0);
            if (!ok) fail(a.status, abort_flag, 42);
            if (ok) {
                ok = mbar_wait_or_abort(&mb_sfree, 0, kWaitBudgetNs, abort_flag);
                if (!ok) fail(a.status, abort_flag, 40);
                else seen = loads;                     // the chain has consumed it (so it landed)
            }
            if (ok) {
                if (n_slots > 1) {
                    ok = load_state(1);
                    if (!ok) fail(a.status, abort_flag, 43);
                } else {
                    ok = final_phase();
                    if (!ok) fail(a.status, abort_flag, 46);
                }
            }
            for (int k = 0; ok && k < n_slots; ++k) {
                if (!mbar_wait_or_abort(&mb_sfree, (k + 1) & 1, kWaitBudgetNs, abort_flag)) { fail(a.status, abort_flag, 41); break; }
                seen = loads;
                int lh, tb, te;
                sch.slot(k, n, lh, tb, te);
                const bool hand_over = sch.is_prefix(k);
                const bool seg_end = kSeg && sch.seg_mode >= 2;   // a segment run's end: hand-over entry me
                if (kSeg && sch.seg_mode == 2) {
                    bulk_store(a.ho_base + (size_t)me * 65536, sm, 65536);   // A: the images the chain wrote
                } else {
                    const bool to_h = hand_over || seg_end;
                    const CUtensorMap* dst = to_h ? &hmap : &smap;
                    const int row = (to_h ? me : lh) * kD;
#pragma unroll
                    for (int b = 0; b < 4; ++b) tma_store_2d(dst, sbuf + 4096 * b, 32 * b, row);
                }
                bulk_commit();
                if (hand_over || seg_end) {
                    bulk_wait0();                      // the state is in global memory ...
                    fence_proxy_async_global();
                    __threadfence();
                    grid_dep_wait();                   // (after the factor kernel's flag reset)
                    ho_store_release(a.ho_flag + me, 1);   // ... before CTA i + 1 may read it
                }
                if (k + 2 <= n_slots) {
                    bulk_wait_read0();                 // slot k's state has left the buffer
                    if (k + 2 < n_slots) {
                        if (!load_state(k + 2)) { fail(a.status, abort_flag, 43); break; }
                    } else if (!final_phase()) {
                        fail(a.status, abort_flag, 46);
                        break;
                    }
                }
            }
            bulk_wait0();                              // every state store is complete
            if (loads > seen) mbar_wait(&mb_st, (loads - 1) & 1, kWaitBudgetNs);   // abort: a load in flight
            if (ca) mbar_wait(&mb_ca, 0, kWaitBudgetNs);   // (A's images have landed)
        }
        __syncwarp();
    } else {
        // =========================================================== state chain (warps 0-15)
        const int q = warp & 3, cgp = warp >> 2;         // TMEM lane quadrant, column group
        const int r = 32 * q + lane;                     // row of S (value index)
        const uint32_t lane_off = (uint32_t)(32 * q) << 16;
        float* sbuf = reinterpret_cast<float*>(sm + SM_SB);   // swizzled rows, see sb_idx
        int st_seen = 0;                                 // mb_st phases waited for (uniform)
        TileCursor cc;                                   // the chain's tile
        cc.init(sch, a);
        const int me = (int)blockIdx.x;
        // K(jj) (TMA tile, buffer jj % 3) in fp32 (exact, and exact in tf32) into the B operand
        // buffer of X.  Called between MMA_X(jj-1), the last reader of the buffer, and the ready
        // signal of tile jj.
        // A chain warp arrives (lane 0, for the warp) on sready / xready / uready / sfree only while
        // every wait of lane 0 has seen its phase complete: the MMA and state warps take a completed
        // phase as proof that the copies the passes waited for have landed (after another role
        // failed, they would otherwise release buffers whose copies may still be in flight).
        bool failed = false;
        auto cwait = [&](uint64_t* bar, uint32_t parity, int where) {
            const bool ok = mbar_wait_or_abort(bar, parity, kWaitBudgetNs, abort_flag);
            if (!ok) { fail(a.status, abort_flag, where); failed = true; }
            return ok;
        };
        // (one arrival per warp: every lane's TMEM stores / shared-memory writes were completed and
        // fenced before the __syncwarp; lane 0 then arrives, a release)
        auto carrive = [&](uint64_t* bar) {
            __syncwarp();
            if (lane == 0 && !failed) mbar_arrive(bar);
        };
        auto make_k32 = [&](int jj) -> bool {
            const bool ok = cwait(&mb_tk[jj % 3], (jj / 3) & 1, 16);
            const uint8_t* kb = sm + SM_K + (jj % 3) * 16384;
            uint8_t* k32 = sm + SM_K32;
#pragma unroll
            for (int u = 0; u < 2; ++u) {                  // 64 rows x 16 chunks of 8 bf16
                const int e = tid + kChain * u;
                const int t = e >> 4, c16 = e & 15, cb = c16 >> 3, c = c16 & 7;
                const uint4 w = *reinterpret_cast<const uint4*>(kb + cb * 8192 + sw128_offset(t, c));
                const uint32_t wv[4] = {w.x, w.y, w.z, w.w};
                uint32_t f[8];
#pragma unroll
                for (int i = 0; i < 4; ++i) {
                    f[2 * i] = wv[i] << 16;
                    f[2 * i + 1] = wv[i] & 0xFFFF0000u;
                }
                // dims 64 cb + 8 c .. + 7: fp32 block 2 cb + c / 4, chunks 2 (c % 4) and 2 (c % 4) + 1
                uint8_t* rowp = k32 + (2 * cb + (c >> 2)) * 8192;
                const int q0 = 2 * (c & 3);
                *reinterpret_cast<uint4*>(rowp + sw128_offset(t, q0)) = make_uint4(f[0], f[1], f[2], f[3]);
                *reinterpret_cast<uint4*>(rowp + sw128_offset(t, q0 + 1)) = make_uint4(f[4], f[5], f[6], f[7]);
            }
            fence_async_smem();                            // generic writes -> the tensor core's reads
            return ok;
        };
        auto rec_consts = [&](int jj) {                    // -gamma[64], gamma_C of tile jj's record
            return reinterpret_cast<const float*>(sm + SM_R + (jj & 1) * kRecSlot + kRecT);
        };
        float den = 0.f;
        // Deferred decay: TMEM holds S~ with the head's state S = sig * S~.  A tile folds its decay
        // gamma_C into sig (the W pass applies sig and u_scale = 1 / (gamma_C sig), so MMA_S
        // accumulates onto S~ with no pass over the state); when sig gamma_C would drop below
        // kSigMin the tile instead writes gamma_C S back into TMEM and sig restarts at 1.
        float sig = 1.f;
        // Write sizes (optional): column t of the U region is u_t scaled by u_scale gamma_C /
        // gamma_t, u_t = beta_t (v_t - alpha_t S_{t-1} k_t) the token's write.  The Ũ pass sums
        // each column's squares over this warp's 32 rows and adds them, rescaled to u_t, into
        // s_u2 (four warps per column); after the next barrier warp 0 takes the square roots and
        // sums them over the tile's tokens into the head's total.
        const bool want_w = a.wnorm != nullptr;
        float wacc = 0.f;                                  // warp 0: the head's running sum
        int prev_lh = -1, prev_slot = -1;
        bool prev_last = false;
        // a head's write-size sum: to hand-over entry i when the slot begins a head shared with
        // CTA i + 1, else (with the first part's sum from entry i - 1 when it ends a head shared
        // with CTA i - 1) to the output; warp 0, lane 0
        auto put_wsum = [&](int slot, int lh, float sum) -> bool {
            if (sch.is_prefix(slot)) {
                a.ho_wsum[me] = sum;
                __threadfence();
                grid_dep_wait();                           // (after the factor kernel's flag reset)
                ho_store_release(a.ho_wflag + me, 1);
                return true;
            }
            if (sch.is_suffix(slot)) {
                grid_dep_wait();                           // (the factor kernel's reset of the flag is complete)
                const uint64_t t0 = global_ns();
                while (ho_load_acquire(a.ho_wflag + me - 1) == 0) {
                    if (*abort_flag || global_ns() - t0 > kWaitBudgetNs) return false;
                    __nanosleep(64);
                }
                sum += *reinterpret_cast<volatile const float*>(a.ho_wsum + me - 1);
            }
            a.wnorm[lh] = sum;
            return true;
        };
        auto fold_writes = [&](int jj) {                   // warp 0: tile jj's sizes into wacc
            float* b = s_u2[jj & 1];
            float sacc = sqrtf(b[lane]) + sqrtf(b[lane + 32]);
            b[lane] = 0.f;
            b[lane + 32] = 0.f;
#pragma unroll
            for (int m = 16; m >= 1; m >>= 1) sacc += __shfl_xor_sync(0xffffffffu, sacc, m);
            wacc += sacc;
        };
        for (int j = 0; j < NJ; ++j) {                     // j: global tile index
            const int lh = cc.lh, jt = cc.jt, slot = cc.k; // head, tile within the head, slot
            const bool last = jt == cc.te - 1;             // the slot's last tile
            if (named_sync_or(2, kChain, *abort_flag)) break;
            cwait(&mb_tr[j & 1], (j >> 1) & 1, 13);
            const float gC = rec_consts(j)[64];
            float w_gamma = 0.f;                           // gamma_t of this lane's column in the Ũ pass
            if (want_w) {
                w_gamma = -rec_consts(j)[16 * cgp + (lane >> 1)];
                if (j > 0 && warp == 0) {
                    fold_writes(j - 1);
                    if (prev_last) {
                        if (lane == 0 && !put_wsum(prev_slot, prev_lh, wacc)) fail(a.status, abort_flag, 44);
                        wacc = 0.f;
                    }
                }
            }

            if (j == 0) {
                // ---- the CTA's first head: its state from the staging buffer into TMEM, as S~
                // (sig = 1) and as S_before, and sum S_before^2
                cwait(&mb_st, 0, 14);
                st_seen = 1;
                float sv[32];
                if (kSeg && sch.seg_mode >= 2) {           // a later segment: from I or from 0
#pragma unroll
                    for (int e = 0; e < 32; ++e) sv[e] = (sch.seg_mode == 2 && r == 32 * cgp + e) ? 1.f : 0.f;
                } else {
#pragma unroll
                    for (int e = 0; e < 8; ++e) {
                        const float4 x = *reinterpret_cast<const float4*>(sbuf + sb_idx(r, 8 * cgp + e));
                        sv[4 * e] = x.x; sv[4 * e + 1] = x.y; sv[4 * e + 2] = x.z; sv[4 * e + 3] = x.w;
                    }
                }
#pragma unroll
                for (int e = 0; e < 32; ++e) den = fmaf(sv[e], sv[e], den);
                carrive(&mb_sfree);                              // the staging buffer has been read
                tmem_st32(tm + lane_off + TM_S + 32 * cgp, sv);
                tmem_st32(tm + lane_off + TM_SB + 32 * cgp, sv);
                make_k32(0);
                tmem_st_wait();
                tc_fence_before();
                carrive(&mb_sready);
            }
            const bool rescale = sig * gC < kSigMin;       // uniform over the CTA
            const float u_scale = rescale ? 1.f : 1.f / (gC * sig);

            // ---- W pass: W^T = V^T - sig X~^T diag(gamma) from the V and X regions (X~ = S~ K^T),
            // scaled by u_scale, (hi, lo) in place over this thread's 16 X columns (tokens 16 cgp ..)
            cwait(&mb_x, j & 1, 10);
            tc_fence_after();
            // read-out: the row decays of the thread's 16 tokens, taken now (the record's slot is
            // released to the next load once MMA_U(j) completes, before the U~ pass)
            float dl[kOut ? 16 : 1];
            if constexpr (kOut) {
                const float* src = rec_consts(j) + kRecConsts + 16 * cgp;
#pragma unroll
                for (int e = 0; e < 4; ++e) {
                    const float4 d4 = *reinterpret_cast<const float4*>(src + 4 * e);
                    dl[4 * e] = d4.x; dl[4 * e + 1] = d4.y; dl[4 * e + 2] = d4.z; dl[4 * e + 3] = d4.w;
                }
            }
            {
                float xv[16], vv[16], cf[16];
                tmem_ld16(tm + lane_off + TM_X + 16 * cgp, xv);
                tmem_ld16(tm + lane_off + TM_V + 16 * cgp, vv);
                const float* gm = rec_consts(j) + 16 * cgp;         // -gamma of the thread's tokens
#pragma unroll
                for (int e = 0; e < 4; ++e) {
                    const float4 g4 = *reinterpret_cast<const float4*>(gm + 4 * e);
                    cf[4 * e] = g4.x * sig; cf[4 * e + 1] = g4.y * sig; cf[4 * e + 2] = g4.z * sig; cf[4 * e + 3] = g4.w * sig;
                }
                tmem_ld_wait();
                if (kSeg && sch.seg_mode == 2) {           // the run that forms a segment's A: v = 0
#pragma unroll
                    for (int e = 0; e < 16; ++e) vv[e] = 0.f;
                }
                uint32_t hi[8], lo[8];
#pragma unroll
                for (int i = 0; i < 8; ++i)
                    split2(fmaf(cf[2 * i], xv[2 * i], vv[2 * i]) * u_scale,
                           fmaf(cf[2 * i + 1], xv[2 * i + 1], vv[2 * i + 1]) * u_scale, hi[i], lo[i]);
                tmem_st8(tm + lane_off + TM_X + 16 * cgp, hi);
                tmem_st8(tm + lane_off + TM_X + 16 * cgp + 8, lo);
                tmem_st_wait();
            }
            tc_fence_before();
            carrive(&mb_xready);

            // ---- while MMA_U runs: rescale S~ if the decay would underflow the deferred scale
            // (MMA_X(j) has read S~; MMA_S(j) waits for uready), and K(j+1) in fp32.  For the
            // read-out, a tile that starts a 128-token block also writes the state before it,
            // sig S~ (row r, columns 32 cgp ..).
            const bool snap = kOut && (jt & 1) == 0;       // uniform over the CTA
            if (rescale || snap) {
                float sv[32];
                tmem_ld32(tm + lane_off + TM_S + 32 * cgp, sv);
                tmem_ld_wait();
                if (snap) {
                    float* dst = a.snap + ((((size_t)lh * a.n_blk + (jt >> 1)) * 32 + 8 * cgp) * kD + r) * 4;
#pragma unroll
                    for (int e = 0; e < 8; ++e)
                        *reinterpret_cast<float4*>(dst + e * kD * 4) =
                            make_float4(sv[4 * e] * sig, sv[4 * e + 1] * sig, sv[4 * e + 2] * sig, sv[4 * e + 3] * sig);
                }
                if (rescale) {
                    const float f = gC * sig;
#pragma unroll
                    for (int e = 0; e < 32; ++e) sv[e] *= f;
                    tmem_st32(tm + lane_off + TM_S + 32 * cgp, sv);
                    tmem_st_wait();
                }
            }
            sig = rescale ? 1.f : gC * sig;                // the deferred decay after tile j
            if (j + 1 < NJ) make_k32(j + 1);

            // ---- U~ pass: (hi, lo) in place over this thread's 16 U columns
            cwait(&mb_u, j & 1, 11);
            tc_fence_after();
            {
                float uv[16];
                tmem_ld16(tm + lane_off + TM_U + 16 * cgp, uv);
                tmem_ld_wait();
                if constexpr (kOut) {
                    // with the record's undecayed T the column is u_t u_scale = u_t / sig: u_t out
                    // for the read-out (tokens jt 64 + 16 cgp .. of row r)
                    float* dst = a.ubuf + ((((size_t)lh * n + jt) * 16 + 4 * cgp) * kD + r) * 4;
#pragma unroll
                    for (int e = 0; e < 4; ++e)
                        *reinterpret_cast<float4*>(dst + e * kD * 4) =
                            make_float4(uv[4 * e] * sig, uv[4 * e + 1] * sig, uv[4 * e + 2] * sig, uv[4 * e + 3] * sig);
                }
                if (want_w) {
                    // squares summed over the warp's 32 rows, column by column: halving exchanges
                    // leave lanes 2c and 2c + 1 with column c (token 16 cgp + c) of the 16
                    float x[16];
#pragma unroll
                    for (int i = 0; i < 16; ++i) x[i] = uv[i] * uv[i];
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
                    // U column -> u_t.  u_scale gamma_C is 1 / sig >= 1 unless the tile restarts
                    // the deferred decay; then it is gamma_C, and below 2^-60 the columns of the
                    // early tokens, scaled by gamma_C / gamma_t, are no longer representable: such
                    // a tile contributes nothing
                    float wf;
                    if constexpr (kOut) {
                        wf = sig;                          // the column is u_t / sig
                    } else {
                        const float sc = u_scale * gC;
                        wf = sc >= 0x1p-60f ? w_gamma / sc : 0.f;
                    }
                    if ((lane & 1) == 0) atomicAdd(&s_u2[j & 1][16 * cgp + (lane >> 1)], x[0] * wf * wf);
                }
                if constexpr (kOut) {
                    // the row decay exp(G_C - G_t) that T~ carries on the path without read-out
#pragma unroll
                    for (int e = 0; e < 16; ++e) uv[e] *= dl[e];
                }
                uint32_t hi[8], lo[8];
#pragma unroll
                for (int i = 0; i < 8; ++i) split2(uv[2 * i], uv[2 * i + 1], hi[i], lo[i]);
                tmem_st8(tm + lane_off + TM_U + 16 * cgp, hi);
                tmem_st8(tm + lane_off + TM_U + 16 * cgp + 8, lo);
                tmem_st_wait();
            }
            tc_fence_before();
            carrive(&mb_uready);
            if (!last) {
                // the next tile of this head may start X as soon as MMA_S(j) is queued
                carrive(&mb_sready);
            } else {
                // ---- head boundary: S_after = sig S~ out through the staging buffer, the next
                // head's state (staged meanwhile) into TMEM, drift partials against S_before
                const bool has_next = j + 1 < NJ;          // uniform
                // a last slot that ends a head begun by CTA i - 1: S_before is not in TMEM (the
                // slot started from the handed-over state) but staged, and its square sum is taken
                // here
                const bool shared_end = sch.is_suffix(slot);
                float den_end = 0.f;
                bool ok = cwait(&mb_s, j & 1, 12);
                if (!cwait(&mb_st, st_seen & 1, 14)) ok = false;
                ok = __all_sync(0xffffffffu, ok) != 0;     // (the pass below is warp-collective)
                ++st_seen;
                tc_fence_after();
                if (kSeg && sch.seg_mode == 1 && ok) {
                    // segment combine: S_0 = sig S~ as bfloat16 (hi, lo) K-major images (row r, this
                    // warp's 32 columns) in the free tile buffers, then S~ = S_0 A + B from the
                    // product and the staged B, sig = 1: the pass below writes S_after and the drift
                    {
                        float sv[32];
                        tmem_ld32(tm + lane_off + TM_S + 32 * cgp, sv);
                        tmem_ld_wait();
#pragma unroll
                        for (int e = 0; e < 32; ++e) sv[e] *= sig;
#pragma unroll
                        for (int c = 0; c < 4; ++c) {
                            uint4 vh, vl;
                            split8(sv + 8 * c, vh, vl);
                            const uint32_t off = (cgp >> 1) * 16384 + sw128_offset(r, 4 * (cgp & 1) + c);
                            *reinterpret_cast<uint4*>(sm + off) = vh;
                            *reinterpret_cast<uint4*>(sm + 32768 + off) = vl;
                        }
                    }
                    fence_async_smem();
                    tc_fence_before();
                    carrive(&mb_cimg);
                    ok = __all_sync(0xffffffffu, cwait(&mb_cd, 0, 17)) != 0;
                    if (ok) {
                        tc_fence_after();
                        float dv[32];
                        tmem_ld32(tm + lane_off + TM_X + 32 * cgp, dv);
                        tmem_ld_wait();
#pragma unroll
                        for (int e = 0; e < 8; ++e) {
                            const float4 b = *reinterpret_cast<const float4*>(sbuf + sb_idx(r, 8 * cgp + e));
                            dv[4 * e] += b.x; dv[4 * e + 1] += b.y; dv[4 * e + 2] += b.z; dv[4 * e + 3] += b.w;
                        }
                        tmem_st32(tm + lane_off + TM_S + 32 * cgp, dv);
                        tmem_st_wait();
                        sig = 1.f;
                    }
                }
                float num = 0.f, den_next = 0.f;
                if (ok) {
#pragma unroll
                    for (int half = 0; half < 2; ++half) {
                        const uint32_t col = 32 * cgp + 16 * half;
                        const int ch = 8 * cgp + 4 * half;     // this half's 16-byte chunks of row r
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
                        if (kSeg && sch.seg_mode == 2) {       // A: row r's (hi, lo) images, MN-major
#pragma unroll
                            for (int c2 = 0; c2 < 2; ++c2) {
                                uint4 vh, vl;
                                split8(sa + 8 * c2, vh, vl);
                                const uint32_t off = (cgp >> 1) * 16384 + sw128_offset(r, 4 * (cgp & 1) + 2 * half + c2);
                                *reinterpret_cast<uint4*>(sm + off) = vh;
                                *reinterpret_cast<uint4*>(sm + 32768 + off) = vl;
                            }
                        }
                    }
                    tmem_st_wait();
                }
                tc_fence_before();
                fence_async_smem();                        // S_after -> the state warp's TMA store
                carrive(&mb_sfree);
                if (has_next) carrive(&mb_sready);               // the next head's state is in TMEM
                // partial sums: pairwise in fp32, over the warp's lanes and then over the 16 warps
                // (the FP64 pipe is far too slow for this path)
                float fn = num, fd = shared_end ? den_end : den;
#pragma unroll
                for (int m = 16; m >= 1; m >>= 1) {
                    fn += __shfl_xor_sync(0xffffffffu, fn, m);
                    fd += __shfl_xor_sync(0xffffffffu, fd, m);
                }
                if (lane == 0) { s_red[0][warp] = fn; s_red[1][warp] = fd; }
                if (named_sync_or(2, kChain, !ok)) break;
                if (warp == 0 && a.partials != nullptr && !sch.is_prefix(slot) && (!kSeg || sch.seg_mode == 1)) {
                    // (a shared head's drift: at its end; a segmented head's: CTA 0's, after the combine)
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
            cc.next(sch, a);
        }
        // the CTA's last tile (always a head's last) once every warp's Ũ pass has added to it
        if (want_w && NJ > 0 && !named_sync_or(2, kChain, *abort_flag) && warp == 0) {
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

// =============================================================================================
// Read-out kernel: o_t = q_scale S_t q_t for every token of the chunk
// =============================================================================================
// Unrolling Eq. 1 from the state S_b before a block of 128 tokens, with G the inclusive cumulative
// log-decay inside the block and u_i = beta_i (v_i - alpha_i S_{i-1} k_i) the write of token i,
//   S_t = exp(G_t) S_b + sum_{i <= t} exp(G_t - G_i) u_i k_i^T,
// so the block's outputs are, at once,
//   O = (P o D) U + diag(exp(G)) Q S_b^T,    P = Q K^T,   D[t][i] = exp(G_t - G_i) for i <= t, else 0,
// with U the rows u_i.  The update kernel leaves u_i and S_b in the workspace; this kernel takes one
// (layer, value head, block) item at a time: P by a bfloat16 MMA (exact inputs) into TMEM, P o D
// (in place) and diag(exp(G)) Q formed in fp32 in TMEM as the A operands of two kind::tf32 MMAs
// that accumulate O, then O q_scale to the output.  Items run one after another on a persistent CTA
// per SM; the next item's Q and K load while O is formed, its U and S_b during the store.
// Warp w serves TMEM lanes 32 (w % 4) .. + 31 (the block's tokens) and column half w / 4.
constexpr int kRoThreads = 256;
constexpr int kRoBlk = 128;                            // tokens per item (two update tiles)
constexpr uint32_t kRoTmemCols = 512;
constexpr uint32_t RT_P = 0, RT_Q = 128, RT_O = 256;  // TMEM: P (then P o D), diag(exp(G)) Q, O
// shared-memory map (bytes from a 1024-aligned base)
constexpr uint32_t RO_Q = 0;        // 32 KB: Q, 2 column blocks (d 0-63, 64-127) x 128 rows x 128 B, SW128
constexpr uint32_t RO_K = 32768;    // 32 KB: K, same layout
constexpr uint32_t RO_U = 65536;    // 64 KB: U, [32 token chunks][d_v][4] fp32 (N = d_v, K = tokens, no swizzle)
constexpr uint32_t RO_S = 131072;   // 64 KB: S_b, [32 d_k chunks][d_v][4] fp32 (N = d_v, K = d_k, no swizzle)
constexpr uint32_t kRoSmemAlloc = 196608 + 1024;

struct RoArgs {
    int L, Hk, Hv, T, n_tiles, n_blk;
    float q_scale;
    const float* g;
    const float* ubuf;       // the update kernel's u_t and block states (TcArgs::ubuf, TcArgs::snap)
    const float* snap;
    __nv_bfloat16* out;
    int32_t* status;
};

__global__ void __launch_bounds__(kRoThreads, 1)
gdn_readout_kernel(const __grid_constant__ CUtensorMap qmap, const __grid_constant__ CUtensorMap kmap, RoArgs a)
{
    extern __shared__ uint8_t smem_raw[];
    uint8_t* sm = smem_raw + ((1024 - (smem_u32(smem_raw) & 1023)) & 1023);
    __shared__ uint64_t mb_qk, mb_us, mb_p, mb_o;
    __shared__ uint32_t s_tmem;
    __shared__ int s_abort;
    __shared__ __align__(16) float s_g2[kRoBlk];      // G log2(e) of the item's tokens
    volatile int* abort_flag = &s_abort;
    grid_dep_launch();
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int items = a.L * a.Hv * a.n_blk;            // item = (layer * Hv + head) * n_blk + block
    if (warp == 0) { tmem_alloc(&s_tmem, kRoTmemCols); tmem_relinquish(); }
    if (tid == 32) {
        mbar_init(&mb_qk, 1); mbar_init(&mb_us, 1); mbar_init(&mb_p, 1); mbar_init(&mb_o, 1);
        fence_barrier_init();
        prefetch_tensormap(&qmap); prefetch_tensormap(&kmap);
        s_abort = 0;
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tm = s_tmem;

    auto load_qk = [&](int it) {                       // thread 0: the item's Q and K blocks
        const int lh = it / a.n_blk, b = it - lh * a.n_blk, l = lh / a.Hv, h = lh - l * a.Hv;
        const int kh = (int)(((long long)h * a.Hk) / a.Hv);
        mbar_arrive_expect_tx(&mb_qk, 4 * 16384);
#pragma unroll
        for (int th = 0; th < 2; ++th) {
#pragma unroll
            for (int cb = 0; cb < 2; ++cb) {
                const uint32_t off = cb * 16384 + th * 8192;
                tma_load_4d(sm + RO_Q + off, &qmap, &mb_qk, 64 * cb, kh, b * kRoBlk + 64 * th, l);
                tma_load_4d(sm + RO_K + off, &kmap, &mb_qk, 64 * cb, kh, b * kRoBlk + 64 * th, l);
            }
        }
    };
    // the item's block has two update tiles, or one (the last block of an odd tile count: its
    // second half of U is zero-filled in shared memory)
    auto block_tiles = [&](int it) { return min(2, a.n_tiles - 2 * (it % a.n_blk)); };
    auto load_us = [&](int it) {                       // thread 0: the item's U and S_b (bulk copies)
        const int lh = it / a.n_blk, b = it - lh * a.n_blk;
        const uint32_t ub = (uint32_t)block_tiles(it) * 32768u;
        mbar_arrive_expect_tx(&mb_us, ub + 65536u);
        bulk_load_tx(sm + RO_U, a.ubuf + ((size_t)lh * a.n_tiles + 2 * b) * 16 * kD * 4, ub, &mb_us);
        bulk_load_tx(sm + RO_S, a.snap + ((size_t)lh * a.n_blk + b) * 32 * kD * 4, 65536u, &mb_us);
    };
    int n_qk = 0, n_us = 0, n_p = 0, n_o = 0;          // copies / MMA groups issued (thread 0 / warp 0)
    const int first = (int)blockIdx.x, G = (int)gridDim.x;
    // q, k and g are inputs of the call; U and S_b are written by the update kernel, which the
    // wait covers
    if (tid == 0 && first < items) { load_qk(first); ++n_qk; }
    grid_dep_wait();
    if (tid == 0 && first < items) { load_us(first); ++n_us; }

    const int q4 = warp & 3, hc = warp >> 2;
    const int t = 32 * q4 + lane;                      // the thread's token row of the block
    const uint32_t lane_off = (uint32_t)(32 * q4) << 16;
    int c = 0;
    for (int it = first; it < items; it += G, ++c) {
        const int lh = it / a.n_blk, b = it - lh * a.n_blk, l = lh / a.Hv, h = lh - l * a.Hv;
        const int nxt = it + G;
        if (warp == 4) {
            // inclusive cumulative log-decay of the block's tokens, four per lane (past T: g = 0)
            float gv[4];
#pragma unroll
            for (int e = 0; e < 4; ++e) {
                const int tok = b * kRoBlk + 4 * lane + e;
                gv[e] = tok < a.T ? a.g[((size_t)l * a.T + tok) * a.Hv + h] : 0.f;
            }
            gv[1] += gv[0]; gv[2] += gv[1]; gv[3] += gv[2];
            float incl = gv[3];
#pragma unroll
            for (int m = 1; m < 32; m <<= 1) {
                const float y = __shfl_up_sync(0xffffffffu, incl, m);
                if (lane >= m) incl += y;
            }
            const float base = incl - gv[3];
            *reinterpret_cast<float4*>(s_g2 + 4 * lane) =
                make_float4((base + gv[0]) * kLog2e, (base + gv[1]) * kLog2e, (base + gv[2]) * kLog2e,
                            (base + gv[3]) * kLog2e);
        }
        if (warp == 0) {                               // P = Q K^T
            uint64_t aq[2][4], bk[2][4];
#pragma unroll
            for (int s = 0; s < 8; ++s) {
                const uint32_t off = (s >> 2) * 16384 + (s & 3) * 32;
                aq[s >> 2][s & 3] = sdesc_sw128(smem_u32(sm + RO_Q + off), 16, 1024);
                bk[s >> 2][s & 3] = sdesc_sw128(smem_u32(sm + RO_K + off), 16, 1024);
            }
            if (c == 0 ? warp_wait(&mb_qk, 0, wait_budget_ns(a.status), abort_flag)   // (the workspace's
                       : warp_wait(&mb_qk, c & 1, kWaitBudgetNs, abort_flag)) {      //  budget: first wait)
                tc_fence_after();
                if (elect_one()) {
                    mma4_bf16_ss_1t(tm + RT_P, aq[0], bk[0], idesc_bf16(128, 128, 0, 0), 0);
                    mma4_bf16_ss_1t(tm + RT_P, aq[1], bk[1], idesc_bf16(128, 128, 0, 0), 1);
                }
                __syncwarp();
                mma_commit(&mb_p);
                ++n_p;
            } else if (lane == 0) {
                fail(a.status, abort_flag, 60);
            }
        }
        bool ok = mbar_wait_or_abort(&mb_p, c & 1, kWaitBudgetNs, abort_flag);
        if (!ok && !*abort_flag) fail(a.status, abort_flag, 61);
        if (__syncthreads_or(!ok)) break;              // (also publishes s_g2)
        tc_fence_after();
        if (block_tiles(it) == 1) {                    // (the previous item's MMAs have read U)
            float4* z = reinterpret_cast<float4*>(sm + RO_U + 32768);
#pragma unroll
            for (int e = 0; e < 8; ++e) z[tid + kRoThreads * e] = make_float4(0.f, 0.f, 0.f, 0.f);
        }
        {
            // P o D in place: columns 64 hc .. + 63 of row t; a 16-column group right of every
            // row of the warp is all zero
            const float g2t = s_g2[t];
#pragma unroll
            for (int k = 0; k < 4; ++k) {
                const int c0 = 64 * hc + 16 * k;
                uint32_t o[16];
                if (c0 <= 32 * q4 + 31) {              // uniform over the warp
                    float p[16];
                    tmem_ld16(tm + lane_off + RT_P + c0, p);
                    tmem_ld_wait();
#pragma unroll
                    for (int e4 = 0; e4 < 4; ++e4) {
                        const float4 gi = *reinterpret_cast<const float4*>(s_g2 + c0 + 4 * e4);
                        const float gg[4] = {gi.x, gi.y, gi.z, gi.w};
#pragma unroll
                        for (int e = 0; e < 4; ++e) {
                            const int i = c0 + 4 * e4 + e;
                            o[4 * e4 + e] = __float_as_uint(i <= t ? p[4 * e4 + e] * fast_exp2(g2t - gg[e]) : 0.f);
                        }
                    }
                } else {
#pragma unroll
                    for (int e = 0; e < 16; ++e) o[e] = 0u;
                }
                tmem_st16(tm + lane_off + RT_P + c0, o);
            }
            // diag(exp(G)) Q: dims 64 hc .. + 63 of row t, from the swizzled bfloat16 block
            const float gam = fast_exp2(g2t);
            const uint8_t* qb = sm + RO_Q + hc * 16384;
#pragma unroll
            for (int k = 0; k < 4; ++k) {
                uint32_t o[16];
#pragma unroll
                for (int h2 = 0; h2 < 2; ++h2) {
                    const uint4 w = *reinterpret_cast<const uint4*>(qb + sw128_offset(t, 2 * k + h2));
                    const uint32_t wv[4] = {w.x, w.y, w.z, w.w};
#pragma unroll
                    for (int i = 0; i < 4; ++i) {
                        o[8 * h2 + 2 * i] = __float_as_uint(__uint_as_float(wv[i] << 16) * gam);
                        o[8 * h2 + 2 * i + 1] = __float_as_uint(__uint_as_float(wv[i] & 0xFFFF0000u) * gam);
                    }
                }
                tmem_st16(tm + lane_off + RT_Q + 64 * hc + 16 * k, o);
            }
            tmem_st_wait();
        }
        fence_async_smem();                            // Q's generic reads before the next TMA write
        tc_fence_before();
        __syncthreads();
        // Q and K have been read (P is complete, diag(exp(G)) Q formed): the next item's blocks
        if (tid == 0 && nxt < items) { load_qk(nxt); ++n_qk; }
        if (warp == 0) {                               // O = (P o D) U + (diag(exp(G)) Q) S_b^T
            uint32_t ap[4][4], aq[4][4];
            uint64_t bu[4][4], bs[4][4];
#pragma unroll
            for (int s = 0; s < 16; ++s) {
                ap[s >> 2][s & 3] = tm + RT_P + 8 * s;
                aq[s >> 2][s & 3] = tm + RT_Q + 8 * s;
                // K = 8 per MMA: two 4-element chunks of 2048 bytes
                bu[s >> 2][s & 3] = sdesc_interleave(smem_u32(sm + RO_U) + 4096 * s, 2048, 128);
                bs[s >> 2][s & 3] = sdesc_interleave(smem_u32(sm + RO_S) + 4096 * s, 2048, 128);
            }
            if (warp_wait(&mb_us, c & 1, kWaitBudgetNs, abort_flag)) {
                tc_fence_after();
                if (elect_one()) {
#pragma unroll
                    for (int g4 = 0; g4 < 4; ++g4) mma4_tf32_ta_1t(tm + RT_O, ap[g4], bu[g4], idesc_tf32(128, 128), g4 != 0);
#pragma unroll
                    for (int g4 = 0; g4 < 4; ++g4) mma4_tf32_ta_1t(tm + RT_O, aq[g4], bs[g4], idesc_tf32(128, 128), 1);
                }
                __syncwarp();
                mma_commit(&mb_o);
                ++n_o;
            } else if (lane == 0) {
                fail(a.status, abort_flag, 62);
            }
        }
        ok = mbar_wait_or_abort(&mb_o, c & 1, kWaitBudgetNs, abort_flag);
        if (!ok && !*abort_flag) fail(a.status, abort_flag, 63);
        if (__syncthreads_or(!ok)) break;
        tc_fence_after();
        // U and S_b have been read: the next item's
        if (tid == 0 && nxt < items) { load_us(nxt); ++n_us; }
        {   // O q_scale -> bfloat16, dims 64 hc .. + 63 of the token's output row
            const int tok = b * kRoBlk + t;
            __nv_bfloat16* dst = a.out + (((size_t)l * a.T + tok) * a.Hv + h) * kD + 64 * hc;
#pragma unroll
            for (int k = 0; k < 4; ++k) {
                float o[16];
                tmem_ld16(tm + lane_off + RT_O + 64 * hc + 16 * k, o);
                tmem_ld_wait();
                if (tok < a.T) {
                    uint32_t w[8];
#pragma unroll
                    for (int i = 0; i < 8; ++i) w[i] = pack_bf16x2(o[2 * i] * a.q_scale, o[2 * i + 1] * a.q_scale);
                    uint4* d4 = reinterpret_cast<uint4*>(dst + 16 * k);
                    d4[0] = make_uint4(w[0], w[1], w[2], w[3]);
                    d4[1] = make_uint4(w[4], w[5], w[6], w[7]);
                }
            }
        }
        tc_fence_before();
        __syncthreads();                               // O has been read
    }
    if (*abort_flag) {
        // after a failure: what this CTA issued lands before TMEM is freed and the CTA ends (at
        // most one phase of each barrier is outstanding)
        if (tid == 0) {
            if (n_qk > 0) mbar_wait(&mb_qk, (n_qk - 1) & 1, kWaitBudgetNs);
            if (n_us > 0) mbar_wait(&mb_us, (n_us - 1) & 1, kWaitBudgetNs);
        }
        if (warp == 0 && lane == 0) {
            if (n_p > 0) mbar_wait(&mb_p, (n_p - 1) & 1, kWaitBudgetNs);
            if (n_o > 0) mbar_wait(&mb_o, (n_o - 1) & 1, kWaitBudgetNs);
        }
    }
    tc_fence_before();
    __syncthreads();
    if (warp == 0) {
        tc_fence_after();
        tmem_dealloc(tm, kRoTmemCols);
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

// fp32 rows [rows][cols] as a 2-D map: a box of 32 columns x 128 rows, 128-byte swizzle; columns
// past `cols` read as zero.
bool make_rows_map(CUtensorMap* map, void* base, long long rows, int cols) {
    EncodeTiledFn enc = encode_fn();
    if (!enc) return false;
    cuuint64_t dims[2] = {(cuuint64_t)cols, (cuuint64_t)rows};
    cuuint64_t strides[1] = {(cuuint64_t)cols * 4};
    cuuint32_t box[2] = {32, (cuuint32_t)kD};
    cuuint32_t es[2] = {1, 1};
    return enc(map, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 2, base, dims, strides, box, es,
               CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
               CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// The state [heads * 128][128] fp32: a box is one column block of one head.
bool make_state_map(CUtensorMap* map, void* base, long long heads) {
    return make_rows_map(map, base, heads * kD, kD);
}

// Scratch: the WY records, then the update kernel's hand-over area for up to one CTA per SM:
// states [grid][128][128] fp32 (1024-aligned), flags [2][grid] int32, write-size sums [grid];
// with the read-out, then each token's write u_t (128 floats per token and value head) and the
// state at the start of every 128-token block (128 x 128 floats per block and value head), both
// 1024-aligned, in the layouts of TcArgs::ubuf and TcArgs::snap.
struct TcScratch {
    size_t rec, ho_state, ho_flags, ho_wsum, ubuf, snap, total;
};

size_t align1k(size_t x) { return (x + 1023) & ~size_t(1023); }

// Segments per head (see ChainSched) for a call without read-out or write sizes: two when three
// CTAs per head fit on the SMs and each half keeps at least 4 tiles (the combine costs a few
// microseconds), else 1 (not segmented: the heads share the SMs).
int segments_for(int heads, int n_tiles, int sms) {
    return ((long long)heads * 3 <= sms && n_tiles >= 8) ? 2 : 1;
}

TcScratch tc_scratch_layout(int L, int Hv, int T, bool out) {
    const int sms = device_sm_count();
    const size_t n_tiles = (size_t)(T + kC - 1) / kC, n_blk = (n_tiles + 1) / 2, heads = (size_t)L * Hv;
    // the chain's grid: one CTA per SM at most, or 2 seg - 1 per head when segmented
    const int sg = out ? 1 : segments_for(L * Hv, (int)n_tiles, sms);
    const int grid = std::max(1, sg > 1 ? L * Hv * (2 * sg - 1) : std::min(L * Hv, sms));
    TcScratch l;
    l.rec = 0;
    l.ho_state = align1k(heads * n_tiles * rec_bytes(out));          // hand-over / segment end states
    l.ho_flags = l.ho_state + (size_t)grid * kD * kD * 4;
    l.ho_wsum = l.ho_flags + 2 * (size_t)grid * 4;
    l.total = l.ho_wsum + (size_t)grid * 4;
    l.ubuf = l.snap = 0;
    if (out) {
        l.ubuf = align1k(l.total);
        l.snap = align1k(l.ubuf + heads * kD * n_tiles * kC * 4);
        l.total = l.snap + heads * n_blk * kD * kD * 4;
    }
    return l;
}

}  // namespace

size_t gdn_tc_scratch_bytes(int L, int Hv, int dk, int dv, int dtype, int T, bool out) {
    if (dk != kD || dv != kD || dtype != DELTAS_BF16 || L <= 0 || Hv <= 0 || T <= 0) return 0;
    return tc_scratch_layout(L, Hv, T, out).total;
}

bool gdn_tc_shape(const GdnArgs& a) {
    return a.dk == kD && a.dv == kD && a.dtype == DELTAS_BF16 && a.T > 0;
}

bool gdn_tc_supported(const GdnArgs& a) {
    const long long n_tiles = (a.T + kC - 1) / kC;
    return gdn_tc_shape(a) &&
           (long long)a.L * a.Hv * kD < (1ll << 31) &&                          // TMA row coordinate
           (long long)a.L * a.Hv * n_tiles < (1ll << 31) &&                     // factor-kernel items
           (long long)a.L * a.Hv * ((n_tiles + 1) / 2) * kD < (1ll << 31) &&    // read-out block rows
           a.scratch != nullptr &&
           a.scratch_bytes >= gdn_tc_scratch_bytes(a.L, a.Hv, a.dk, a.dv, a.dtype, a.T, a.out != nullptr) &&
           encode_fn() != nullptr;
}

cudaError_t launch_gdn_update_tc(const GdnArgs& a, cudaStream_t s) {
    const bool out = a.out != nullptr;
    const TcScratch sl = tc_scratch_layout(a.L, a.Hv, a.T, out);   // hand-over space for device_sm_count() CTAs
    // one chain CTA per SM that this context may use (a CTA waits at its end for its neighbour's
    // hand-over, so the grid must not exceed what can be resident)
    const int sms = context_sm_count();
    const int n_tiles = (a.T + kC - 1) / kC, n_blk = (n_tiles + 1) / 2;
    const long long heads = (long long)a.L * a.Hv;
    // few heads: each head's tiles in segments on 2 seg - 1 CTAs (not with the read-out or the write
    // sizes: a later segment's run does not see the true state)
    const int sg = (out || a.wnorm != nullptr) ? 1 : segments_for(a.L * a.Hv, n_tiles, sms);
    const int grid = sg > 1 ? a.L * a.Hv * (2 * sg - 1) : std::min(a.L * a.Hv, sms);
    CUtensorMap kmap, vmap, smap, hmap, qmap;
    if (!make_map(&kmap, a.k, a.L, a.T, a.Hk) || !make_map(&vmap, a.v, a.L, a.T, a.Hv) ||
        !make_state_map(&smap, a.state, heads) || !make_state_map(&hmap, a.scratch + sl.ho_state, grid))
        return cudaErrorInvalidValue;
    if (out && !make_map(&qmap, a.q, a.L, a.T, a.Hk)) return cudaErrorInvalidValue;
    auto chain = out ? gdn_update_tc_kernel<true, false>
                     : sg > 1 ? gdn_update_tc_kernel<false, true> : gdn_update_tc_kernel<false, false>;
    {   // set on every launch (cheap, and right for whichever device and context is current)
        cudaError_t e = cudaFuncSetAttribute(chain, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kSmemAlloc);
        if (e == cudaSuccess)
            e = cudaFuncSetAttribute(gdn_wy_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kWySmemAlloc);
        if (e == cudaSuccess && out)
            e = cudaFuncSetAttribute(gdn_readout_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                     (int)kRoSmemAlloc);

        if (e != cudaSuccess) return e;
    }
    // factor kernel: one record per (layer, value head, tile), kWyCtasPerSm persistent CTAs per SM
    WyArgs w;
    w.L = a.L; w.Hk = a.Hk; w.Hv = a.Hv; w.T = a.T; w.n_tiles = n_tiles; w.out = out ? 1 : 0;
    w.g = a.g; w.beta = a.beta; w.rec = a.scratch; w.status = a.status;
    w.ho_flags = reinterpret_cast<int32_t*>(a.scratch + sl.ho_flags);
    w.n_ho_flags = 2 * grid;
    const long long items = heads * n_tiles;
    const int wgrid = (int)std::min<long long>(items, (long long)sms * kWyCtasPerSm);
    gdn_wy_kernel<<<wgrid, kWyThreads, kWySmemAlloc, s>>>(kmap, w);
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return e;
    // update kernel: one persistent CTA per SM (the kernel needs the whole SM: 512 TMEM columns,
    // ~211 KB of shared memory); each takes every grid-th head, or an equal run of tiles
    TcArgs t;
    t.L = a.L; t.Hk = a.Hk; t.Hv = a.Hv; t.T = a.T; t.n_tiles = n_tiles;
    t.state = a.state; t.partials = a.partials; t.wnorm = a.wnorm; t.rec = a.scratch; t.status = a.status;
    t.ho_flag = reinterpret_cast<int32_t*>(a.scratch + sl.ho_flags);
    t.ho_wflag = t.ho_flag + grid;
    t.ho_wsum = reinterpret_cast<float*>(a.scratch + sl.ho_wsum);
    t.seg = sg;
    t.ho_base = a.scratch + sl.ho_state;
    t.ubuf = out ? reinterpret_cast<float*>(a.scratch + sl.ubuf) : nullptr;
    t.snap = out ? reinterpret_cast<float*>(a.scratch + sl.snap) : nullptr;
    t.n_blk = n_blk;
    // equal tile runs, with heads split between neighbouring CTAs, when they shorten the slowest
    // CTA: a boundary between slots costs about 0.45 of a tile and the hand-over about three
    // tiles (measured: 512- and 1024-token chunks gain 5-6 %, chunks of 2-3 tiles lose)
    t.split = 0;
    const int H = a.L * a.Hv;
    if (sg == 1 && H > grid && H % grid != 0) {
        const double whole = std::ceil((double)H / grid) * (n_tiles + 0.45);
        const double runs = std::ceil((double)H * n_tiles / grid);
        const double parted = runs + (runs / n_tiles + 2.0) * 0.45 + 3.0;
        t.split = parted < whole ? 1 : 0;
    }
    e = launch_dependent(chain, dim3(grid), dim3(kThreads), (size_t)kSmemAlloc, s, kmap, vmap, smap, hmap, t);
    if (e != cudaSuccess) return e;
    if (!out) return e;
    // read-out kernel: one persistent CTA per SM over the (layer, value head, 128-token block) items;
    // its CTAs take the SMs the update kernel leaves free and wait there for its results
    RoArgs r;
    r.L = a.L; r.Hk = a.Hk; r.Hv = a.Hv; r.T = a.T; r.n_tiles = n_tiles; r.n_blk = n_blk; r.q_scale = a.q_scale;
    r.g = a.g; r.ubuf = t.ubuf; r.snap = t.snap; r.out = static_cast<__nv_bfloat16*>(a.out); r.status = a.status;
    const int rgrid = (int)std::min<long long>(heads * n_blk, sms);
    return launch_dependent(gdn_readout_kernel, dim3(rgrid), dim3(kRoThreads), (size_t)kRoSmemAlloc, s, qmap, kmap, r);
}

}  // namespace deltas
