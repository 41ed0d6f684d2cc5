// Per-head retain selection for the cache-internal token signals of Sec. 4.3 (key norm -||k||,
// value norm ||v||, one score per token and KV head): the Sec. 3.3 rule -- sink, window, N
// temporal spans over the candidates' arrival chunks with a quota each, then a fill from the best
// remaining candidates -- applied to every (layer, KV head) plane with the slots' own scores.
//
// A cluster of kHeadCluster 1024-thread CTAs ranks one plane, each CTA a contiguous quarter of
// its candidates (the first also the sink, the last the window).  After each step the CTAs add
// up their partial counts through distributed shared memory, and every CTA takes the same
// decisions from the sums:
//   1. the smallest / largest candidate chunk and score key (block reductions, then over the
//      cluster; negative chunk ids are reported);
//   2. every candidate's span and its 56-bit key: the score's IEEE total-order bits (32) above
//      the complement of the slot (24 bits, so that the earlier slot ranks higher on equal
//      scores).  Keys are unique.  The 32-bit score part and the span (one byte) of every
//      candidate are kept in shared memory when the plane fits, else in the workspace; the slot
//      part is the candidate's index.  The same pass counts the spans and builds the quota
//      select's first-digit histogram;
//   3. quota: for every span with more candidates than the quota q, a radix select (8-bit
//      digits, most significant first, starting at the highest bit in which two candidates'
//      keys differ, all spans in one pass over the candidates) narrows a key prefix until the
//      candidates at or above it are exactly the span's best q: a span is done as soon as the
//      digit bin it stops in is taken whole, so distinct scores resolve within the score digits
//      and the slot digits are read only for exact ties;
//   4. fill: the same select over the candidates the quota left, as one group, for the
//      remaining capacity R - kept (its first-digit histogram built by the pass that marks the
//      quota's choices);
//   5. emit: every warp owns a contiguous stretch of its CTA's slots; it counts its kept slots,
//      the CTAs' totals and a scan of the 32 warp counts give its offset, and it writes its kept
//      slots in order (retain_idx ascending) and the mask.
// Nothing is sorted: the cost is a fixed number of passes over the plane's candidates.
#include <algorithm>
#include <climits>

#include "internal.cuh"

namespace deltas {
namespace {

constexpr int kHeadThreads = 1024;
constexpr int kHeadWarps = kHeadThreads / 32;
constexpr int kHeadMaxSpans = 32;
constexpr int kSlotBits = 24;                         // slots < 2^20 (DELTAS_SELECT_MAX_CACHE_LEN)
constexpr uint32_t kSlotMask = (1u << kSlotBits) - 1u;
constexpr size_t kHeadSmemLimit = 220 * 1024;         // dynamic shared memory the kernel may ask for
constexpr int kUnroll = 4;                            // candidates per lane per pass iteration
constexpr int kHeadCluster = 4;                       // CTAs per plane (one cluster)

enum HeadMode : int { kKeepAll = 0, kKeepNone = 1, kKeepSome = 2 };

struct HeadArgs {
    int M, n_s, n_w, N;            // N >= 1 (0 is read as one span)
    int n_planes, cache_len, plane_stride;
    const int32_t* tok_chunk;      // [n_planes][plane_stride]
    const float* tok_score;        // [n_planes][plane_stride]
    int32_t* retain_idx;           // [n_planes][M]
    int32_t* n_retained;
    uint8_t* mask;                 // [n_planes][plane_stride] or null
    uint32_t* ws_keys;             // [n_planes][cache_len] when the keys do not fit in shared memory
    uint8_t* ws_spans;             // [n_planes][cache_len]
    int keys_in_smem;
    int slice;                     // candidates per CTA of a plane's cluster
    int32_t* status;
};

__host__ __device__ inline size_t align256(size_t x) { return (x + 255) & ~size_t(255); }

__device__ __forceinline__ uint32_t score_order_bits(float s) {
    const uint32_t b = __float_as_uint(s);
    return (b & 0x80000000u) ? ~b : (b | 0x80000000u);
}

// 56-bit key of candidate c (slot lo + c): larger = better.
__device__ __forceinline__ uint64_t cand_key(const uint32_t* keys, int c, int lo) {
    return ((uint64_t)keys[c] << kSlotBits) | (uint64_t)(kSlotMask - (uint32_t)(lo + c));
}

// (key(c) >> shift) >= prefix, in 32-bit arithmetic while the shift stays within the slot bits'
// reach (the usual case: distinct scores resolve before the slot digits).
__device__ __forceinline__ bool key_at_least(const uint32_t* keys, int c, int lo, int shift, uint64_t prefix) {
    if (shift >= kSlotBits) return (uint64_t)(keys[c] >> (shift - kSlotBits)) >= prefix;
    return (cand_key(keys, c, lo) >> shift) >= prefix;
}

// Per-group state of a block-wide radix select (shared memory).  A group j with mode kKeepSome
// keeps the candidates c with (key(c) >> shift[j]) >= prefix[j]; `target` counts how many are
// still to be found below the current prefix.
struct RadixGroups {
    uint64_t prefix[kHeadMaxSpans];
    int shift[kHeadMaxSpans];
    int target[kHeadMaxSpans];
    int mode[kHeadMaxSpans];
    int done[kHeadMaxSpans];
};

// Adds one to hist[bin] for every lane with bin >= 0.  When the warp's active lanes share one
// bin (the common case in the first digits, where most keys agree) a single atomic adds them all.
__device__ __forceinline__ void hist_add(unsigned* hist, int bin, int lane) {
    const unsigned act = __ballot_sync(0xffffffffu, bin >= 0);
    if (act == 0) return;
    const int leader = __ffs(act) - 1;
    const int b0 = __shfl_sync(0xffffffffu, bin, leader);
    if (__all_sync(0xffffffffu, bin < 0 || bin == b0)) {
        if (lane == leader) atomicAdd(&hist[b0], (unsigned)__popc(act));
    } else if (bin >= 0) {
        atomicAdd(&hist[bin], 1u);
    }
}

// ---- the plane's cluster: kHeadCluster CTAs, each ranking a quarter of the candidates.  Every
// phase ends with a cluster barrier after which each CTA reads its peers' partial results from
// their shared memory and combines them the same way, so every CTA takes the same decisions.  The
// barriers stand at the top level of the kernel or of loops whose trip counts come from those
// combined results: every thread of every CTA passes the same sequence of them.

__device__ __forceinline__ uint32_t cluster_rank() {
    uint32_t r;
    asm volatile("mov.u32 %0, %%cluster_ctarank;" : "=r"(r));
    return r;
}
// arrive (release: this CTA's shared-memory writes become visible to the cluster) and wait for
// every thread of every CTA of the cluster (acquire)
__device__ __forceinline__ void cluster_barrier() {
    asm volatile("barrier.cluster.arrive.release.aligned;\n\tbarrier.cluster.wait.acquire.aligned;" ::: "memory");
}
// the word at `p` (this CTA's shared memory) in CTA `rank` of the cluster
__device__ __forceinline__ uint32_t peer_word(const void* p, uint32_t rank) {
    const uint32_t local = (uint32_t)__cvta_generic_to_shared(p);
    uint32_t remote, v;
    asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(remote) : "r"(local), "r"(rank));
    asm volatile("ld.shared::cluster.u32 %0, [%1];" : "=r"(v) : "r"(remote) : "memory");
    return v;
}
// stores v at `p` (this CTA's shared memory) in CTA `rank` of the cluster
__device__ __forceinline__ void peer_store(void* p, uint32_t rank, uint32_t v) {
    const uint32_t local = (uint32_t)__cvta_generic_to_shared(p);
    uint32_t remote;
    asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(remote) : "r"(local), "r"(rank));
    asm volatile("st.shared::cluster.u32 [%0], %1;" :: "r"(remote), "r"(v) : "memory");
}
// Every warp-wide access to a peer names one CTA for all its lanes: lanes of one instruction that
// address different CTAs measured about ten times slower.
// out[e] = the sum over the cluster's CTAs of their local[e], e < n (integer sums: any order)
__device__ __forceinline__ void cluster_sum(const unsigned* local, unsigned* out, int n) {
    for (int e = threadIdx.x; e < n; e += kHeadThreads) {
        unsigned v[kHeadCluster];
#pragma unroll
        for (int r = 0; r < kHeadCluster; ++r) v[r] = peer_word(local + e, (uint32_t)r);
        unsigned t = 0;
#pragma unroll
        for (int r = 0; r < kHeadCluster; ++r) t += v[r];
        out[e] = t;
    }
}

__device__ __forceinline__ int first_digit_width(int top_bits) { return min(8, top_bits); }

// Radix select for G groups at once over the 56-bit keys of this CTA's m candidates (local index
// c: key bits keys[c], slot base + c), whose bits above `top_bits` are `top_prefix` for every
// candidate of the plane (so the digits start at the highest bit in which two candidates differ).
// group_of(c) returns the candidate's group, or -1 when it takes no part.  Digits are 8 bits (the
// last one narrower), most significant first.  On entry hsum holds the cluster's histogram of the
// first digit, summed from the local histograms in buffer `buf` of hloc (two buffers of bstride
// words, the first G * 256 of each used); every later
// digit is counted locally into the other buffer, summed over the cluster after a barrier, and
// scanned by every CTA alike.  A local buffer is cleared only two digits after it was counted: by
// then every peer has read it (it was summed before the barrier of the digit in between).  On
// return `buf` is the buffer counted last, every group with mode kKeepSome has its (prefix, shift),
// and every CTA holds the same group state.
template <typename GroupOf>
__device__ void radix_select(const uint32_t* keys, int m, int base, int G, int bstride, int top_bits,
                             uint64_t top_prefix, RadixGroups& rg, unsigned* hloc, unsigned* hsum, int& buf,
                             int* s_open, GroupOf group_of)
{
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    for (int j = threadIdx.x; j < G; j += kHeadThreads) {
        rg.prefix[j] = top_prefix;
        rg.shift[j] = top_bits;
        rg.done[j] = rg.mode[j] != kKeepSome;
    }
    __syncthreads();
    if (threadIdx.x == 0) {
        int open = 0;
        for (int j = 0; j < G; ++j) open += rg.done[j] ? 0 : 1;
        *s_open = open;
    }
    __syncthreads();
    int bits = top_bits;
    bool have = true;
    while (bits > 0 && *s_open > 0) {
        const int w = min(8, bits), shift = bits - w;
        const uint64_t dmask = (1ull << w) - 1ull;
        if (!have) {
            buf ^= 1;
            unsigned* hist = hloc + (size_t)buf * bstride;
            for (int e = threadIdx.x; e < G * 256; e += kHeadThreads) hist[e] = 0;
            __syncthreads();
            // kUnroll candidates per lane and iteration: their loads are independent and overlap
            for (int c00 = warp * 32 * kUnroll; c00 < m; c00 += kHeadThreads * kUnroll) {
                int bin[kUnroll];
#pragma unroll
                for (int u = 0; u < kUnroll; ++u) {
                    const int c = c00 + u * 32 + lane;
                    bin[u] = -1;
                    if (c < m) {
                        const int j = group_of(c);
                        if (j >= 0 && !rg.done[j]) {
                            if (shift >= kSlotBits) {            // score digits: 32-bit arithmetic
                                const uint32_t k = keys[c];
                                const int hs = bits - kSlotBits;
                                const bool match = hs >= 32 || (uint64_t)(k >> hs) == rg.prefix[j];
                                if (match) bin[u] = j * 256 + (int)((k >> (shift - kSlotBits)) & (uint32_t)dmask);
                            } else {
                                const uint64_t key = cand_key(keys, c, base);
                                if ((key >> bits) == rg.prefix[j]) bin[u] = j * 256 + (int)((key >> shift) & dmask);
                            }
                        }
                    }
                }
#pragma unroll
                for (int u = 0; u < kUnroll; ++u) hist_add(hist, bin[u], lane);
            }
            cluster_barrier();                         // every CTA's count of this digit is complete
            cluster_sum(hist, hsum, G * 256);
            __syncthreads();
        }
        have = false;
        // one warp per open group: lane l holds digits 255-8l .. 248-8l (descending across lanes)
        for (int j = warp; j < G; j += kHeadWarps) {
            if (rg.done[j]) continue;
            const unsigned* hj = hsum + j * 256;
            unsigned local = 0;
#pragma unroll
            for (int e = 0; e < 8; ++e) local += hj[255 - 8 * lane - e];
            unsigned incl = local;
#pragma unroll
            for (int mm = 1; mm < 32; mm <<= 1) {
                const unsigned y = __shfl_up_sync(0xffffffffu, incl, mm);
                if (lane >= mm) incl += y;
            }
            const unsigned target = (unsigned)rg.target[j];
            const unsigned excl = incl - local;
            const bool mine = excl < target && target <= incl;
            const unsigned who = __ballot_sync(0xffffffffu, mine);
            if (mine && lane == __ffs(who) - 1) {
                unsigned above = excl;
                int d = 255 - 8 * lane;
                for (int e = 0; e < 8; ++e, --d) {
                    const unsigned h = hj[d];
                    if (above + h >= target) break;
                    above += h;
                }
                const int need = (int)(target - above);           // 1 <= need <= hist[d]
                rg.prefix[j] = (rg.prefix[j] << w) | (uint64_t)d;
                rg.shift[j] = shift;
                rg.target[j] = need;
                if ((unsigned)need == hj[d]) {                    // the bin is taken whole
                    rg.done[j] = 1;
                    atomicSub(s_open, 1);
                }
            }
        }
        __syncthreads();
        bits = shift;
    }
}

// Exclusive scan of the 32 per-warp counts in s_cnt (in place); returns the total.
__device__ int scan_warp_counts(int* s_cnt, int* s_total) {
    if (threadIdx.x < 32) {
        const int v = s_cnt[threadIdx.x];
        int x = v;
#pragma unroll
        for (int m = 1; m < 32; m <<= 1) {
            const int y = __shfl_up_sync(0xffffffffu, x, m);
            if ((int)threadIdx.x >= m) x += y;
        }
        s_cnt[threadIdx.x] = x - v;
        if (threadIdx.x == 31) *s_total = x;
    }
    __syncthreads();
    return *s_total;
}

__global__ void __cluster_dims__(kHeadCluster, 1, 1) __launch_bounds__(kHeadThreads, 1)
select_heads_kernel(HeadArgs a)
{
    extern __shared__ uint4 smem_raw[];
    __shared__ RadixGroups rg;
    __shared__ unsigned s_cnt[kHeadMaxSpans], s_cnt_all[kHeadMaxSpans];     // span counts: own, cluster
    __shared__ int s_min, s_max, s_bad, s_open, s_total, s_fill;
    __shared__ unsigned s_kmin, s_kmax;
    __shared__ int g_min, g_max, g_bad;
    __shared__ unsigned g_kmin, g_kmax;
    __shared__ long long s_thr[kHeadMaxSpans];
    __shared__ int s_warp[kHeadWarps];
    __shared__ int s_kept_all[kHeadCluster];              // every CTA's kept count, pushed by each

    const int p = blockIdx.x / kHeadCluster;
    const int rank = (int)cluster_rank();
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int T = a.cache_len;
    const int32_t* tok_chunk = a.tok_chunk + (size_t)p * a.plane_stride;
    const float* tok_score = a.tok_score + (size_t)p * a.plane_stride;
    int32_t* out = a.retain_idx + (size_t)p * a.M;
    uint8_t* mask = a.mask ? a.mask + (size_t)p * a.plane_stride : nullptr;

    grid_dep_wait();                                   // the scores of the last append are written
    if (T <= a.M) {                                    // nothing to evict: the identity
        const int i0 = (int)((long long)T * rank / kHeadCluster), i1 = (int)((long long)T * (rank + 1) / kHeadCluster);
        for (int i = i0 + tid; i < i1; i += kHeadThreads) {
            out[i] = i;
            if (mask) mask[i] = 1;
        }
        if (p == 0 && rank == 0 && tid == 0) *a.n_retained = T;
        return;                                        // (no CTA of the cluster reads a peer)
    }
    const int lo = a.n_s, hi = T - a.n_w, n_cand = hi - lo;
    const int R = a.M - a.n_s - a.n_w, N = a.N, q = R / N;
    // this CTA's candidates [c0, c1) and its slots [s0, s1) (the plane's sink goes to the first CTA,
    // its window to the last): the slices tile the plane in order
    const int c0 = min(n_cand, rank * a.slice), c1 = min(n_cand, c0 + a.slice), m = c1 - c0;
    const int s0 = rank == 0 ? 0 : lo + c0, s1 = rank == kHeadCluster - 1 ? T : lo + c1;
    const int base = lo + c0;                          // slot of local candidate 0

    // ---- 1. candidate chunk range and score-key range; every chunk id must be >= 0
    if (tid == 0) { s_min = INT_MAX; s_max = INT_MIN; s_bad = 0; s_kmin = 0xffffffffu; s_kmax = 0u; }
    if (tid < kHeadMaxSpans) s_cnt[tid] = 0;
    __syncthreads();
    // Slot b0 + 1024 u + lane for warp-uniform b0 (phases 1 and 2 alike).  When the CTA's slots fit in
    // one round (4096), phase 1's loads stay in registers for phase 2.
    const bool held = s1 - s0 <= 4 * kHeadThreads;
    int h_ch[4] = {0, 0, 0, 0};
    float h_sc[4] = {0.f, 0.f, 0.f, 0.f};
    {
        int mn = INT_MAX, mx = INT_MIN, bad = 0;
        unsigned kmin = 0xffffffffu, kmax = 0u;
        for (int b0 = s0 + 32 * warp; b0 < s1; b0 += 4 * kHeadThreads) {
#pragma unroll
            for (int u = 0; u < 4; ++u) {                  // eight independent loads in flight
                const int i = b0 + u * kHeadThreads + lane;
                h_ch[u] = i < s1 ? tok_chunk[i] : 0;
                h_sc[u] = (i < s1 && i >= lo && i < hi) ? tok_score[i] : 0.f;
            }
#pragma unroll
            for (int u = 0; u < 4; ++u) {
                const int i = b0 + u * kHeadThreads + lane;
                bad |= h_ch[u] < 0;
                if (i < s1 && i >= lo && i < hi) {
                    mn = min(mn, h_ch[u]); mx = max(mx, h_ch[u]);
                    const uint32_t k = score_order_bits(h_sc[u]);
                    kmin = min(kmin, k); kmax = max(kmax, k);
                }
            }
        }
#pragma unroll
        for (int mm = 16; mm >= 1; mm >>= 1) {
            mn = min(mn, __shfl_xor_sync(0xffffffffu, mn, mm));
            mx = max(mx, __shfl_xor_sync(0xffffffffu, mx, mm));
            bad |= __shfl_xor_sync(0xffffffffu, bad, mm);
            kmin = min(kmin, __shfl_xor_sync(0xffffffffu, kmin, mm));
            kmax = max(kmax, __shfl_xor_sync(0xffffffffu, kmax, mm));
        }
        if (lane == 0) {
            atomicMin(&s_min, mn); atomicMax(&s_max, mx); if (bad) atomicOr(&s_bad, 1);
            atomicMin(&s_kmin, kmin); atomicMax(&s_kmax, kmax);
        }
    }
    cluster_barrier();                                 // (1) every CTA's ranges are complete
    if (tid == 0) {                                    // the plane's ranges, CTA by CTA
        uint32_t v[kHeadCluster][5];
#pragma unroll
        for (int r = 0; r < kHeadCluster; ++r) {       // all loads first
            v[r][0] = peer_word(&s_min, r); v[r][1] = peer_word(&s_max, r); v[r][2] = peer_word(&s_bad, r);
            v[r][3] = peer_word(&s_kmin, r); v[r][4] = peer_word(&s_kmax, r);
        }
        int mn = INT_MAX, mx = INT_MIN, bad = 0;
        unsigned kmin = 0xffffffffu, kmax = 0u;
#pragma unroll
        for (int r = 0; r < kHeadCluster; ++r) {
            mn = min(mn, (int)v[r][0]); mx = max(mx, (int)v[r][1]); bad |= (int)v[r][2];
            kmin = min(kmin, v[r][3]); kmax = max(kmax, v[r][4]);
        }
        g_min = mn; g_max = mx; g_bad = bad; g_kmin = kmin; g_kmax = kmax;
    }
    __syncthreads();
    // span(a) = floor((a - c_lo) * N / (c_hi - c_lo + 1)) >= j  <=>  a >= c_lo + ceil(j * len / N):
    // the N - 1 span starts, so that a candidate's span is a search instead of a 64-bit division
    if (tid > 0 && tid < N) {
        const long long len = (long long)g_max - g_min + 1;
        s_thr[tid] = (long long)g_min + ((long long)tid * len + N - 1) / N;
    }
    // the digits start at the highest key bit in which two candidates differ: within the score
    // bits, or within the slot bits when every candidate has the same score
    int top_bits;
    uint64_t top_prefix;
    {
        const uint32_t diff = g_kmin ^ g_kmax;
        if (diff == 0) { top_bits = kSlotBits; top_prefix = g_kmin; }
        else {
            const int hb = 31 - __clz(diff);
            top_bits = kSlotBits + hb + 1;
            top_prefix = (uint64_t)(g_kmin >> hb) >> 1;
        }
    }
    const int dw1 = first_digit_width(top_bits), shift1 = top_bits - dw1;
    const uint64_t dmask1 = (1ull << dw1) - 1ull;

    // ---- 2. keys and spans of this CTA's candidates, span counts, and the quota's first-digit
    // histogram (local buffer 0)
    uint32_t* keys;
    uint8_t* spans;
    unsigned* hloc;                                    // [2][N * 256] local histograms
    if (a.keys_in_smem) {
        keys = reinterpret_cast<uint32_t*>(smem_raw);
        spans = reinterpret_cast<uint8_t*>(keys + a.slice);
        hloc = reinterpret_cast<unsigned*>(smem_raw) + ((size_t)a.slice * 5 + 15) / 16 * 4;
    } else {
        keys = a.ws_keys + (size_t)p * a.cache_len + c0;
        spans = a.ws_spans + (size_t)p * a.cache_len + c0;
        hloc = reinterpret_cast<unsigned*>(smem_raw);
    }
    unsigned* hsum = hloc + 2 * (size_t)N * 256;       // [N * 256] the cluster's sums
    for (int e = tid; e < 2 * N * 256; e += kHeadThreads) hloc[e] = 0;
    __syncthreads();
    for (int b0 = s0 + 32 * warp; b0 < s1; b0 += 4 * kHeadThreads) {   // (warp-uniform trip count)
        int ch[4];
        float sc[4];
#pragma unroll
        for (int u = 0; u < 4; ++u) {                      // phase 1's registers, or all loads first
            const int i = b0 + u * kHeadThreads + lane;
            const bool cand = i < s1 && i >= lo && i < hi;
            ch[u] = held ? h_ch[u] : (cand ? tok_chunk[i] : 0);
            sc[u] = held ? h_sc[u] : (cand ? tok_score[i] : 0.f);
        }
        int jj[4], bin[4];
#pragma unroll
        for (int u = 0; u < 4; ++u) {
            const int i = b0 + u * kHeadThreads + lane;
            const int c = i - base;                        // local candidate index
            jj[u] = -1;
            bin[u] = -1;
            if (i < s1 && i >= lo && i < hi) {
                const uint32_t k = score_order_bits(sc[u]);
                int l = 0, h = N - 1;                      // largest j in [1, N) with ch >= start j
                while (l < h) {
                    const int mid = (l + h + 1) >> 1;
                    if ((long long)ch[u] >= s_thr[mid]) l = mid; else h = mid - 1;
                }
                jj[u] = l;
                keys[c] = k;
                spans[c] = (uint8_t)l;
                const uint64_t key = ((uint64_t)k << kSlotBits) | (uint64_t)(kSlotMask - (uint32_t)(base + c));
                bin[u] = l * 256 + (int)((key >> shift1) & dmask1);
            }
        }
#pragma unroll
        for (int u = 0; u < 4; ++u) {
            hist_add(s_cnt, jj[u], lane);
            hist_add(hloc, bin[u], lane);
        }
    }
    cluster_barrier();                                 // (2) every CTA's counts are complete; the
                                                       // ranges of (1) have been read by every peer
    if (g_bad) {                                       // outputs unspecified; report and stop (every
        if (rank == 0 && tid == 0) record_status(a.status, DELTAS_ERR_DEVICE_INDEX, p);   // CTA alike)
        return;
    }
    cluster_sum(s_cnt, s_cnt_all, N);
    cluster_sum(hloc, hsum, N * 256);
    __syncthreads();

    // ---- 3. quota per span
    if (tid < N) {
        const int cnt = (int)s_cnt_all[tid];
        rg.mode[tid] = cnt <= q ? kKeepAll : (q == 0 ? kKeepNone : kKeepSome);
        rg.target[tid] = q;
    }
    __syncthreads();
    int buf = 0;
    radix_select(keys, m, base, N, N * 256, top_bits, top_prefix, rg, hloc, hsum, buf, &s_open,
                 [&](int c) -> int { return (int)spans[c]; });
    auto kept1 = [&](int c) -> bool {
        const int j = spans[c] & 0x3f;
        const int md = rg.mode[j];
        if (md == kKeepAll) return true;
        if (md == kKeepNone) return false;
        return key_at_least(keys, c, base, rg.shift[j], rg.prefix[j]);
    };

    // ---- 4. fill: the remaining capacity from the best candidates the quota left.  The fill's
    // select reuses the group state, so the quota's outcome is first kept in the span byte
    // (bit 7 = kept by the quota; spans use bits 0..4); the same pass counts the fill's first
    // digit over the candidates left, into the local buffer the quota counted into first-but-last
    // (every peer has read it before the quota's last barrier).
    if (tid == 0) {
        int kept = 0;
        for (int j = 0; j < N; ++j) kept += min(q, (int)s_cnt_all[j]);
        s_fill = R - kept;                             // < the candidates left, since n_cand > R
    }
    unsigned* hfill = hloc + (size_t)(buf ^ 1) * N * 256;
    for (int e = tid; e < 256; e += kHeadThreads) hfill[e] = 0;
    __syncthreads();
    const int fill = s_fill;
    if (fill > 0) {
        for (int c00 = warp * 32 * kUnroll; c00 < m; c00 += kHeadThreads * kUnroll) {
            int bin[kUnroll];
#pragma unroll
            for (int u = 0; u < kUnroll; ++u) {
                const int c = c00 + u * 32 + lane;
                bin[u] = -1;
                if (c < m) {
                    if (kept1(c)) spans[c] |= 0x80u;
                    else bin[u] = (int)((cand_key(keys, c, base) >> shift1) & dmask1);
                }
            }
#pragma unroll
            for (int u = 0; u < kUnroll; ++u) hist_add(hfill, bin[u], lane);
        }
        cluster_barrier();                             // (3) every CTA's fill count is complete
        cluster_sum(hfill, hsum, 256);
        if (tid == 0) { rg.mode[0] = kKeepSome; rg.target[0] = fill; }
        __syncthreads();                               // (every kept1() has read the quota's state)
        // the fill's histograms live in the first 256 words of each local buffer; its first
        // digit is in buffer buf ^ 1, and its next digit goes to the quota's last buffer, which
        // every peer has read before barrier (3)
        buf ^= 1;
        radix_select(keys, m, base, 1, N * 256, top_bits, top_prefix, rg, hloc, hsum, buf, &s_open,
                     [&](int c) -> int { return (spans[c] & 0x80u) ? -1 : 0; });
    }
    const uint64_t fill_prefix = rg.prefix[0];
    const int fill_shift = rg.shift[0];
    auto keep_slot = [&](int i) -> bool {
        if (i < lo || i >= hi) return true;
        const int c = i - base;
        if (fill <= 0) return kept1(c);
        if (spans[c] & 0x80u) return true;
        return key_at_least(keys, c, base, fill_shift, fill_prefix);
    };

    // ---- 5. emit in slot order: this CTA writes its slots [s0, s1) after the kept slots of the
    // CTAs before it; warp w owns a contiguous stretch of them.  The first pass counts and leaves
    // each candidate's decision in bit 6 of its span byte for the second.
    const int n_sl = s1 - s0;
    const int seg = ((n_sl + kHeadWarps - 1) / kHeadWarps + 31) & ~31;
    const int w0 = s0 + min(n_sl, warp * seg), w1 = s0 + min(n_sl, warp * seg + seg);
    int mine = 0;
    for (int i0 = w0; i0 < w1; i0 += 32) {
        const int i = i0 + lane;
        const bool k = i < w1 && keep_slot(i);
        if (k && i >= lo && i < hi) spans[i - base] |= 0x40u;
        mine += __popc(__ballot_sync(0xffffffffu, k));
    }
    if (lane == 0) s_warp[warp] = mine;
    __syncthreads();
    const int cta_kept = scan_warp_counts(s_warp, &s_total);
    if (tid == 0)                                      // into slot `rank` of every CTA's table
        for (int r = 0; r < kHeadCluster; ++r) peer_store(&s_kept_all[rank], r, (uint32_t)cta_kept);
    cluster_barrier();                                 // (4) every CTA's kept count is known; after
                                                       // this no CTA reads or writes a peer
    int s_base = 0, s_all = 0;
#pragma unroll
    for (int r = 0; r < kHeadCluster; ++r) { s_base += r < rank ? s_kept_all[r] : 0; s_all += s_kept_all[r]; }
    int off = s_base + s_warp[warp];
    for (int i0 = w0; i0 < w1; i0 += 32) {
        const int i = i0 + lane;
        const bool k = i < w1 && (i < lo || i >= hi || (spans[i - base] & 0x40u));
        const unsigned b = __ballot_sync(0xffffffffu, k);
        const int at = off + __popc(b & ((1u << lane) - 1u));
        if (k && at < a.M) out[at] = i;
        if (mask && i < w1) mask[i] = k ? 1 : 0;
        off += __popc(b);
    }
    if (rank == 0 && tid == 0) {
        if (s_all != a.M) record_status(a.status, DELTAS_ERR_DEVICE_INDEX, p);   // cannot happen
        if (p == 0) *a.n_retained = min(s_all, a.M);
    }
}

}  // namespace

// Dynamic shared memory of one CTA: its slice's keys and span bytes (when they are kept there),
// two local histogram buffers and the cluster's sums, N x 256 words each.
size_t select_heads_smem_bytes(int slice, int N, bool keys_in_smem) {
    const size_t hist = 3 * (size_t)(N < 1 ? 1 : N) * 256 * sizeof(unsigned);
    return (keys_in_smem ? ((size_t)slice * 5 + 15) / 16 * 16 : 0) + hist;
}

size_t select_heads_workspace_bytes(int n_planes, int cache_len) {
    const size_t n = (size_t)n_planes * (size_t)(cache_len > 0 ? cache_len : 1);
    return kStatusBytes + align256(n * sizeof(uint32_t)) + align256(n);
}

cudaError_t launch_select_heads(const deltas_policy& pol, int n_planes, int cache_len, int plane_stride,
                                const int32_t* tok_chunk, const float* tok_score, int32_t* retain_idx,
                                int32_t* n_retained, uint8_t* mask, void* ws, int32_t* status, cudaStream_t s)
{
    if (n_planes <= 0) return cudaSuccess;
    HeadArgs a;
    a.M = pol.budget_M; a.n_s = pol.n_sink; a.n_w = pol.n_window; a.N = pol.n_buckets < 1 ? 1 : pol.n_buckets;
    a.n_planes = n_planes; a.cache_len = cache_len; a.plane_stride = plane_stride;
    a.tok_chunk = tok_chunk; a.tok_score = tok_score; a.retain_idx = retain_idx; a.n_retained = n_retained;
    a.mask = mask;
    char* w = static_cast<char*>(ws) + kStatusBytes;
    const size_t n = (size_t)n_planes * (size_t)(cache_len > 0 ? cache_len : 1);
    a.ws_keys = reinterpret_cast<uint32_t*>(w);
    a.ws_spans = reinterpret_cast<uint8_t*>(w + align256(n * sizeof(uint32_t)));
    a.status = status;
    const int n_cand = std::max(0, cache_len - a.n_s - a.n_w);
    a.slice = std::max(1, (n_cand + kHeadCluster - 1) / kHeadCluster);
    a.keys_in_smem = select_heads_smem_bytes(a.slice, a.N, true) <= kHeadSmemLimit;
    const size_t smem = select_heads_smem_bytes(a.slice, a.N, a.keys_in_smem != 0);
    // set on every launch (cheap, and right for whichever device and context is current)
    const cudaError_t e = cudaFuncSetAttribute(select_heads_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                               (int)kHeadSmemLimit);
    if (e != cudaSuccess) return e;
    if ((long long)n_planes * kHeadCluster > INT_MAX) return cudaErrorInvalidValue;
    return launch_dependent(select_heads_kernel, dim3(n_planes * kHeadCluster), dim3(kHeadThreads), smem, s, a);
}

}  // namespace deltas
