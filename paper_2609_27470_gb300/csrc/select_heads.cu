// Per-head retain selection for the cache-internal token signals of Sec. 4.3 (key norm -||k||,
// value norm ||v||, one score per token and KV head): the Sec. 3.3 rule -- sink, window, N
// temporal spans over the candidates' arrival chunks with a quota each, then a fill from the best
// remaining candidates -- applied to every (layer, KV head) plane with the slots' own scores.
//
// One 1024-thread CTA ranks one plane:
//   1. the smallest / largest candidate chunk and score key (block reduction; negative chunk ids
//      are reported);
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
//   5. emit: every warp owns a contiguous stretch of slots; it counts its kept slots, a scan of
//      the 32 counts gives its offset, and it writes its kept slots in order (retain_idx
//      ascending) and the mask.
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

// Radix select for G groups at once over the candidates' 56-bit keys, whose bits above
// `top_bits` are `top_prefix` for every candidate (so the digits start at the highest bit in
// which two candidates differ).  group_of(c) returns the candidate's group, or -1 when it takes no
// part.  Digits are 8 bits (the last one narrower), most significant first; two histogram buffers
// alternate so that clearing the next one overlaps the scan of the current one.  `prebuilt`: the
// caller has already filled buffer 0 with the first digit's histogram (while it had every
// candidate in hand anyway), and buffer 1 is zero.  On return every group with mode kKeepSome has
// its (prefix, shift).
__device__ __forceinline__ int first_digit_width(int top_bits) { return min(8, top_bits); }

template <typename GroupOf>
__device__ void radix_select(const uint32_t* keys, int n_cand, int lo, int G, int top_bits, uint64_t top_prefix,
                             RadixGroups& rg, unsigned* hist2, int* s_open, bool prebuilt, GroupOf group_of)
{
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    for (int j = threadIdx.x; j < G; j += kHeadThreads) {
        rg.prefix[j] = top_prefix;
        rg.shift[j] = top_bits;
        rg.done[j] = rg.mode[j] != kKeepSome;
    }
    if (!prebuilt)
        for (int e = threadIdx.x; e < 2 * G * 256; e += kHeadThreads) hist2[e] = 0;
    __syncthreads();
    if (threadIdx.x == 0) {
        int open = 0;
        for (int j = 0; j < G; ++j) open += rg.done[j] ? 0 : 1;
        *s_open = open;
    }
    __syncthreads();
    int bits = top_bits, buf = 0;
    bool have = prebuilt;
    while (bits > 0 && *s_open > 0) {
        const int w = min(8, bits), shift = bits - w;
        const uint64_t dmask = (1ull << w) - 1ull;
        unsigned* hist = hist2 + (size_t)buf * G * 256;
        unsigned* next = hist2 + (size_t)(buf ^ 1) * G * 256;
        // kUnroll candidates per lane and iteration: their loads are independent and overlap
        for (int base = warp * 32 * kUnroll; base < n_cand && !have; base += kHeadThreads * kUnroll) {
            int bin[kUnroll];
#pragma unroll
            for (int u = 0; u < kUnroll; ++u) {
                const int c = base + u * 32 + lane;
                bin[u] = -1;
                if (c < n_cand) {
                    const int j = group_of(c);
                    if (j >= 0 && !rg.done[j]) {
                        if (shift >= kSlotBits) {                // score digits: 32-bit arithmetic
                            const uint32_t k = keys[c];
                            const int hs = bits - kSlotBits;
                            const bool match = hs >= 32 || (uint64_t)(k >> hs) == rg.prefix[j];
                            if (match) bin[u] = j * 256 + (int)((k >> (shift - kSlotBits)) & (uint32_t)dmask);
                        } else {
                            const uint64_t key = cand_key(keys, c, lo);
                            if ((key >> bits) == rg.prefix[j]) bin[u] = j * 256 + (int)((key >> shift) & dmask);
                        }
                    }
                }
            }
#pragma unroll
            for (int u = 0; u < kUnroll; ++u) hist_add(hist, bin[u], lane);
        }
        have = false;
        __syncthreads();
        for (int e = threadIdx.x; e < G * 256; e += kHeadThreads) next[e] = 0;
        // one warp per open group: lane l holds digits 255-8l .. 248-8l (descending across lanes)
        for (int j = warp; j < G; j += kHeadWarps) {
            if (rg.done[j]) continue;
            const unsigned* hj = hist + j * 256;
            unsigned local = 0;
#pragma unroll
            for (int e = 0; e < 8; ++e) local += hj[255 - 8 * lane - e];
            unsigned incl = local;
#pragma unroll
            for (int m = 1; m < 32; m <<= 1) {
                const unsigned y = __shfl_up_sync(0xffffffffu, incl, m);
                if (lane >= m) incl += y;
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
        buf ^= 1;
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

__global__ void __launch_bounds__(kHeadThreads, 1)
select_heads_kernel(HeadArgs a)
{
    extern __shared__ uint4 smem_raw[];
    __shared__ RadixGroups rg;
    __shared__ int s_cnt[kHeadMaxSpans];
    __shared__ int s_min, s_max, s_bad, s_open, s_total, s_fill;
    __shared__ unsigned s_kmin, s_kmax;
    __shared__ long long s_thr[kHeadMaxSpans];
    __shared__ int s_warp[kHeadWarps];

    const int p = blockIdx.x;
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int T = a.cache_len;
    const int32_t* tok_chunk = a.tok_chunk + (size_t)p * a.plane_stride;
    const float* tok_score = a.tok_score + (size_t)p * a.plane_stride;
    int32_t* out = a.retain_idx + (size_t)p * a.M;
    uint8_t* mask = a.mask ? a.mask + (size_t)p * a.plane_stride : nullptr;

    grid_dep_wait();                                   // the scores of the last append are written
    if (T <= a.M) {                                    // nothing to evict: the identity
        for (int i = tid; i < T; i += kHeadThreads) {
            out[i] = i;
            if (mask) mask[i] = 1;
        }
        if (p == 0 && tid == 0) *a.n_retained = T;
        return;
    }
    const int lo = a.n_s, hi = T - a.n_w, n_cand = hi - lo;
    const int R = a.M - a.n_s - a.n_w, N = a.N, q = R / N;

    // ---- 1. candidate chunk range and score-key range; every chunk id must be >= 0
    if (tid == 0) { s_min = INT_MAX; s_max = INT_MIN; s_bad = 0; s_kmin = 0xffffffffu; s_kmax = 0u; }
    if (tid < kHeadMaxSpans) s_cnt[tid] = 0;
    __syncthreads();
    {
        int mn = INT_MAX, mx = INT_MIN, bad = 0;
        unsigned kmin = 0xffffffffu, kmax = 0u;
        for (int i0 = tid; i0 < T; i0 += 4 * kHeadThreads) {
            int c[4];
            float sc[4];
#pragma unroll
            for (int u = 0; u < 4; ++u) {                  // eight independent loads in flight
                const int i = i0 + u * kHeadThreads;
                c[u] = i < T ? tok_chunk[i] : 0;
                sc[u] = (i >= lo && i < hi) ? tok_score[i] : 0.f;
            }
#pragma unroll
            for (int u = 0; u < 4; ++u) {
                const int i = i0 + u * kHeadThreads;
                bad |= c[u] < 0;
                if (i >= lo && i < hi) {
                    mn = min(mn, c[u]); mx = max(mx, c[u]);
                    const uint32_t k = score_order_bits(sc[u]);
                    kmin = min(kmin, k); kmax = max(kmax, k);
                }
            }
        }
#pragma unroll
        for (int m = 16; m >= 1; m >>= 1) {
            mn = min(mn, __shfl_xor_sync(0xffffffffu, mn, m));
            mx = max(mx, __shfl_xor_sync(0xffffffffu, mx, m));
            bad |= __shfl_xor_sync(0xffffffffu, bad, m);
            kmin = min(kmin, __shfl_xor_sync(0xffffffffu, kmin, m));
            kmax = max(kmax, __shfl_xor_sync(0xffffffffu, kmax, m));
        }
        if (lane == 0) {
            atomicMin(&s_min, mn); atomicMax(&s_max, mx); if (bad) atomicOr(&s_bad, 1);
            atomicMin(&s_kmin, kmin); atomicMax(&s_kmax, kmax);
        }
    }
    __syncthreads();
    if (s_bad) {                                       // outputs unspecified; report and stop
        if (tid == 0) record_status(a.status, DELTAS_ERR_DEVICE_INDEX, p);
        return;
    }
    // span(a) = floor((a - c_lo) * N / (c_hi - c_lo + 1)) >= j  <=>  a >= c_lo + ceil(j * len / N):
    // the N - 1 span starts, so that a candidate's span is a search instead of a 64-bit division
    if (tid > 0 && tid < N) {
        const long long len = (long long)s_max - s_min + 1;
        s_thr[tid] = (long long)s_min + ((long long)tid * len + N - 1) / N;
    }
    // the digits start at the highest key bit in which two candidates differ: within the score
    // bits, or within the slot bits when every candidate has the same score
    int top_bits;
    uint64_t top_prefix;
    {
        const uint32_t diff = s_kmin ^ s_kmax;
        if (diff == 0) { top_bits = kSlotBits; top_prefix = s_kmin; }
        else {
            const int hb = 31 - __clz(diff);
            top_bits = kSlotBits + hb + 1;
            top_prefix = (uint64_t)(s_kmin >> hb) >> 1;
        }
    }
    const int dw1 = first_digit_width(top_bits), shift1 = top_bits - dw1;
    const uint64_t dmask1 = (1ull << dw1) - 1ull;

    // ---- 2. keys and spans of the candidates, span counts, and the quota's first-digit histogram
    uint32_t* keys;
    uint8_t* spans;
    unsigned* hist;
    if (a.keys_in_smem) {
        keys = reinterpret_cast<uint32_t*>(smem_raw);
        spans = reinterpret_cast<uint8_t*>(keys + n_cand);
        hist = reinterpret_cast<unsigned*>(smem_raw) + ((size_t)n_cand * 5 + 15) / 16 * 4;   // 2 x N x 256
    } else {
        keys = a.ws_keys + (size_t)p * a.cache_len;
        spans = a.ws_spans + (size_t)p * a.cache_len;
        hist = reinterpret_cast<unsigned*>(smem_raw);
    }
    for (int e = tid; e < 2 * N * 256; e += kHeadThreads) hist[e] = 0;
    __syncthreads();
    for (int base = warp * 32 * kUnroll; base < n_cand; base += kHeadThreads * kUnroll) {
        int ch[kUnroll];
        float sc[kUnroll];
#pragma unroll
        for (int u = 0; u < kUnroll; ++u) {                // all loads first
            const int c = base + u * 32 + lane;
            ch[u] = c < n_cand ? tok_chunk[lo + c] : 0;
            sc[u] = c < n_cand ? tok_score[lo + c] : 0.f;
        }
        int jj[kUnroll], bin[kUnroll];
#pragma unroll
        for (int u = 0; u < kUnroll; ++u) {
            const int c = base + u * 32 + lane;
            jj[u] = -1;
            bin[u] = -1;
            if (c < n_cand) {
                const uint32_t k = score_order_bits(sc[u]);
                int l = 0, h = N - 1;                      // largest j in [1, N) with ch >= start j
                while (l < h) {
                    const int mid = (l + h + 1) >> 1;
                    if ((long long)ch[u] >= s_thr[mid]) l = mid; else h = mid - 1;
                }
                jj[u] = l;
                keys[c] = k;
                spans[c] = (uint8_t)l;
                const uint64_t key = ((uint64_t)k << kSlotBits) | (uint64_t)(kSlotMask - (uint32_t)(lo + c));
                bin[u] = l * 256 + (int)((key >> shift1) & dmask1);
            }
        }
#pragma unroll
        for (int u = 0; u < kUnroll; ++u) {
            hist_add(reinterpret_cast<unsigned*>(s_cnt), jj[u], lane);
            hist_add(hist, bin[u], lane);
        }
    }
    __syncthreads();

    // ---- 3. quota per span
    if (tid < N) {
        const int cnt = s_cnt[tid];
        rg.mode[tid] = cnt <= q ? kKeepAll : (q == 0 ? kKeepNone : kKeepSome);
        rg.target[tid] = q;
    }
    __syncthreads();
    radix_select(keys, n_cand, lo, N, top_bits, top_prefix, rg, hist, &s_open, true,
                 [&](int c) -> int { return (int)spans[c]; });
    auto kept1 = [&](int c) -> bool {
        const int j = spans[c] & 0x3f;
        const int m = rg.mode[j];
        if (m == kKeepAll) return true;
        if (m == kKeepNone) return false;
        return key_at_least(keys, c, lo, rg.shift[j], rg.prefix[j]);
    };

    // ---- 4. fill: the remaining capacity from the best candidates the quota left.  The fill's
    // select reuses the group state, so the quota's outcome is first kept in the span byte
    // (bit 7 = kept by the quota; spans use bits 0..4); the same pass builds the fill's first
    // digit histogram over the candidates left.
    if (tid == 0) {
        int kept = 0;
        for (int j = 0; j < N; ++j) kept += min(q, s_cnt[j]);
        s_fill = R - kept;                             // < the candidates left, since n_cand > R
    }
    for (int e = tid; e < 2 * 256; e += kHeadThreads) hist[e] = 0;
    __syncthreads();
    const int fill = s_fill;
    if (fill > 0) {
        for (int base = warp * 32 * kUnroll; base < n_cand; base += kHeadThreads * kUnroll) {
            int bin[kUnroll];
#pragma unroll
            for (int u = 0; u < kUnroll; ++u) {
                const int c = base + u * 32 + lane;
                bin[u] = -1;
                if (c < n_cand) {
                    if (kept1(c)) spans[c] |= 0x80u;
                    else bin[u] = (int)((cand_key(keys, c, lo) >> shift1) & dmask1);
                }
            }
#pragma unroll
            for (int u = 0; u < kUnroll; ++u) hist_add(hist, bin[u], lane);
        }
        __syncthreads();                               // every kept1() has read the quota's state
        if (tid == 0) { rg.mode[0] = kKeepSome; rg.target[0] = fill; }
        __syncthreads();
        radix_select(keys, n_cand, lo, 1, top_bits, top_prefix, rg, hist, &s_open, true,
                     [&](int c) -> int { return (spans[c] & 0x80u) ? -1 : 0; });
    }
    const uint64_t fill_prefix = rg.prefix[0];
    const int fill_shift = rg.shift[0];
    auto keep_slot = [&](int i) -> bool {
        if (i < lo || i >= hi) return true;
        const int c = i - lo;
        if (fill <= 0) return kept1(c);
        if (spans[c] & 0x80u) return true;
        return key_at_least(keys, c, lo, fill_shift, fill_prefix);
    };

    // ---- 5. emit in slot order: warp w owns slots [w * seg, (w + 1) * seg).  The first pass
    // counts and leaves each candidate's decision in bit 6 of its span byte for the second.
    const int seg = ((T + kHeadWarps - 1) / kHeadWarps + 31) & ~31;
    const int w0 = min(T, warp * seg), w1 = min(T, w0 + seg);
    int mine = 0;
    for (int i0 = w0; i0 < w1; i0 += 32) {
        const int i = i0 + lane;
        const bool k = i < w1 && keep_slot(i);
        if (k && i >= lo && i < hi) spans[i - lo] |= 0x40u;
        mine += __popc(__ballot_sync(0xffffffffu, k));
    }
    if (lane == 0) s_warp[warp] = mine;
    __syncthreads();
    const int total = scan_warp_counts(s_warp, &s_total);
    int off = s_warp[warp];
    for (int i0 = w0; i0 < w1; i0 += 32) {
        const int i = i0 + lane;
        const bool k = i < w1 && (i < lo || i >= hi || (spans[i - lo] & 0x40u));
        const unsigned b = __ballot_sync(0xffffffffu, k);
        const int at = off + __popc(b & ((1u << lane) - 1u));
        if (k && at < a.M) out[at] = i;
        if (mask && i < w1) mask[i] = k ? 1 : 0;
        off += __popc(b);
    }
    if (tid == 0) {
        if (total != a.M) record_status(a.status, DELTAS_ERR_DEVICE_INDEX, p);   // cannot happen
        if (p == 0) *a.n_retained = min(total, a.M);
    }
}

}  // namespace

size_t select_heads_smem_bytes(int n_cand, int N, bool keys_in_smem) {
    const size_t hist = 2 * (size_t)(N < 1 ? 1 : N) * 256 * sizeof(unsigned);
    return (keys_in_smem ? ((size_t)n_cand * 5 + 15) / 16 * 16 : 0) + hist;
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
    a.keys_in_smem = select_heads_smem_bytes(n_cand, a.N, true) <= kHeadSmemLimit;
    const size_t smem = select_heads_smem_bytes(n_cand, a.N, a.keys_in_smem != 0);
    // set on every launch (cheap, and right for whichever device and context is current)
    const cudaError_t e = cudaFuncSetAttribute(select_heads_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                               (int)kHeadSmemLimit);
    if (e != cudaSuccess) return e;
    return launch_dependent(select_heads_kernel, dim3(n_planes), dim3(kHeadThreads), smem, s, a);
}

}  // namespace deltas
