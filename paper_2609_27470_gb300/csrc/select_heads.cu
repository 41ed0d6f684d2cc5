// Per-head retain selection for the cache-internal token signals of Sec. 4.3 (key norm -||k||,
// value norm ||v||, one score per token and KV head): the Sec. 3.3 rule -- sink, window, N
// temporal spans over the candidates' arrival chunks with a quota each, then a fill from the best
// remaining candidates -- applied to every (layer, KV head) plane with the slots' own scores.
//
// One 1024-thread CTA ranks one plane:
//   1. the smallest / largest candidate chunk (block reduction; negative chunk ids are reported);
//   2. every candidate's span and its 56-bit key: the score's IEEE total-order bits (32) above
//      the complement of the slot (24 bits, so that the earlier slot ranks higher on equal
//      scores).  Keys are unique.  The 32-bit score part and the span (one byte) of every
//      candidate are kept in shared memory when the plane fits, else in the workspace; the slot
//      part is the candidate's index;
//   3. quota: for every span with more candidates than the quota q, a radix select (8-bit
//      digits, most significant first, all spans in one pass over the candidates) narrows a key
//      prefix until the candidates at or above it are exactly the span's best q: a span is done
//      as soon as the digit bin it stops in is taken whole, so random scores resolve within the
//      four score digits and the slot digits are read only for exact ties;
//   4. fill: the same select over the candidates the quota left, as one group, for the
//      remaining capacity R - kept;
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
constexpr int kKeyBits = 32 + kSlotBits;
constexpr uint32_t kSlotMask = (1u << kSlotBits) - 1u;
constexpr size_t kHeadSmemLimit = 220 * 1024;         // dynamic shared memory the kernel may ask for

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

// Radix select for G groups at once.  group_of(c) returns the candidate's group, or -1 when the
// candidate takes no part.  On return every group with mode kKeepSome has its (prefix, shift).
template <typename GroupOf>
__device__ void radix_select(const uint32_t* keys, int n_cand, int lo, int G, RadixGroups& rg, unsigned* hist,
                             int* s_remaining, GroupOf group_of)
{
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    for (int j = threadIdx.x; j < G; j += kHeadThreads) {
        rg.prefix[j] = 0;
        rg.shift[j] = kKeyBits;
        rg.done[j] = rg.mode[j] != kKeepSome;
    }
    __syncthreads();
    for (int shift = kKeyBits - 8; shift >= 0; shift -= 8) {
        if (threadIdx.x == 0) {
            int left = 0;
            for (int j = 0; j < G; ++j) left += rg.done[j] ? 0 : 1;
            *s_remaining = left;
        }
        for (int e = threadIdx.x; e < G * 256; e += kHeadThreads) hist[e] = 0;
        __syncthreads();
        if (*s_remaining == 0) break;
        for (int base = warp * 32; base < n_cand; base += kHeadThreads) {
            const int c = base + lane;
            int bin = -1;
            if (c < n_cand) {
                const int j = group_of(c);
                if (j >= 0 && !rg.done[j]) {
                    const uint64_t key = cand_key(keys, c, lo);
                    if ((key >> (shift + 8)) == rg.prefix[j]) bin = j * 256 + (int)((key >> shift) & 255u);
                }
            }
            const unsigned act = __ballot_sync(0xffffffffu, bin >= 0);
            if (bin >= 0) {
                const unsigned peers = __match_any_sync(act, bin);
                if (lane == __ffs(peers) - 1) atomicAdd(&hist[bin], (unsigned)__popc(peers));
            }
        }
        __syncthreads();
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
                rg.prefix[j] = (rg.prefix[j] << 8) | (uint64_t)d;
                rg.shift[j] = shift;
                rg.target[j] = need;
                rg.done[j] = (unsigned)need == hj[d];           // the bin is taken whole
            }
        }
        __syncthreads();
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

__global__ void __launch_bounds__(kHeadThreads)
select_heads_kernel(HeadArgs a)
{
    extern __shared__ uint4 smem_raw[];
    __shared__ RadixGroups rg;
    __shared__ int s_cnt[kHeadMaxSpans];
    __shared__ int s_min, s_max, s_bad, s_remaining, s_total, s_fill_mode;
    __shared__ int s_warp[kHeadWarps];
    __shared__ uint64_t s_fill_prefix;
    __shared__ int s_fill_shift;

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

    // ---- 1. candidate chunk range; every chunk id must be >= 0
    if (tid == 0) { s_min = INT_MAX; s_max = INT_MIN; s_bad = 0; }
    __syncthreads();
    {
        int mn = INT_MAX, mx = INT_MIN, bad = 0;
        for (int i = tid; i < T; i += kHeadThreads) {
            const int c = tok_chunk[i];
            bad |= c < 0;
            if (i >= lo && i < hi) { mn = min(mn, c); mx = max(mx, c); }
        }
#pragma unroll
        for (int m = 16; m >= 1; m >>= 1) {
            mn = min(mn, __shfl_xor_sync(0xffffffffu, mn, m));
            mx = max(mx, __shfl_xor_sync(0xffffffffu, mx, m));
            bad |= __shfl_xor_sync(0xffffffffu, bad, m);
        }
        if (lane == 0) { atomicMin(&s_min, mn); atomicMax(&s_max, mx); if (bad) atomicOr(&s_bad, 1); }
    }
    if (tid < kHeadMaxSpans) s_cnt[tid] = 0;
    __syncthreads();
    if (s_bad) {                                       // outputs unspecified; report and stop
        if (tid == 0) record_status(a.status, DELTAS_ERR_DEVICE_INDEX, p);
        return;
    }
    const int c_lo = s_min;
    const long long span_len = (long long)s_max - c_lo + 1;

    // ---- 2. keys and spans of the candidates, span counts
    uint32_t* keys;
    uint8_t* spans;
    unsigned* hist;
    if (a.keys_in_smem) {
        keys = reinterpret_cast<uint32_t*>(smem_raw);
        spans = reinterpret_cast<uint8_t*>(keys + n_cand);
        hist = reinterpret_cast<unsigned*>(smem_raw) + ((size_t)n_cand * 5 + 15) / 16 * 4;
    } else {
        keys = a.ws_keys + (size_t)p * a.cache_len;
        spans = a.ws_spans + (size_t)p * a.cache_len;
        hist = reinterpret_cast<unsigned*>(smem_raw);
    }
    for (int base = warp * 32; base < n_cand; base += kHeadThreads) {
        const int c = base + lane;
        int j = -1;
        if (c < n_cand) {
            const int i = lo + c;
            j = (int)(((long long)(tok_chunk[i] - c_lo) * N) / span_len);
            keys[c] = score_order_bits(tok_score[i]);
            spans[c] = (uint8_t)j;
        }
        const unsigned act = __ballot_sync(0xffffffffu, j >= 0);
        if (j >= 0) {
            const unsigned peers = __match_any_sync(act, j);
            if (lane == __ffs(peers) - 1) atomicAdd(&s_cnt[j], __popc(peers));
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
    radix_select(keys, n_cand, lo, N, rg, hist, &s_remaining,
                 [&](int c) -> int { return (int)spans[c]; });
    auto kept1 = [&](int c) -> bool {
        const int j = spans[c];
        const int m = rg.mode[j];
        if (m == kKeepAll) return true;
        if (m == kKeepNone) return false;
        return (cand_key(keys, c, lo) >> rg.shift[j]) >= rg.prefix[j];
    };

    // ---- 4. fill: the remaining capacity from the best candidates the quota left.  The fill's
    // select reuses the group state, so the quota's outcome is first kept in the span byte
    // (bit 7 = kept by the quota; spans use bits 0..4).
    for (int c = tid; c < n_cand; c += kHeadThreads)
        if (kept1(c)) spans[c] |= 0x80u;
    __syncthreads();
    if (tid == 0) {
        int kept = 0;
        for (int j = 0; j < N; ++j) kept += min(q, s_cnt[j]);
        const int fill = R - kept;                     // < the candidates left, since n_cand > R
        s_fill_mode = fill > 0 ? kKeepSome : kKeepNone;
        rg.mode[0] = s_fill_mode;
        rg.target[0] = fill;
    }
    __syncthreads();
    if (s_fill_mode == kKeepSome)
        radix_select(keys, n_cand, lo, 1, rg, hist, &s_remaining,
                     [&](int c) -> int { return (spans[c] & 0x80u) ? -1 : 0; });
    if (tid == 0) { s_fill_prefix = rg.prefix[0]; s_fill_shift = rg.shift[0]; }
    __syncthreads();
    const bool fill_on = s_fill_mode == kKeepSome;
    const uint64_t fill_prefix = s_fill_prefix;
    const int fill_shift = s_fill_shift;
    auto keep_slot = [&](int i) -> bool {
        if (i < lo || i >= hi) return true;
        const int c = i - lo;
        if (spans[c] & 0x80u) return true;
        return fill_on && (cand_key(keys, c, lo) >> fill_shift) >= fill_prefix;
    };

    // ---- 5. emit in slot order: warp w owns slots [w * seg, (w + 1) * seg)
    const int seg = ((T + kHeadWarps - 1) / kHeadWarps + 31) & ~31;
    const int w0 = min(T, warp * seg), w1 = min(T, w0 + seg);
    int mine = 0;
    for (int i0 = w0; i0 < w1; i0 += 32) {
        const int i = i0 + lane;
        mine += __popc(__ballot_sync(0xffffffffu, i < w1 && keep_slot(i)));
    }
    if (lane == 0) s_warp[warp] = mine;
    __syncthreads();
    const int total = scan_warp_counts(s_warp, &s_total);
    int off = s_warp[warp];
    for (int i0 = w0; i0 < w1; i0 += 32) {
        const int i = i0 + lane;
        const bool k = i < w1 && keep_slot(i);
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
    const size_t hist = (size_t)(N < 1 ? 1 : N) * 256 * sizeof(unsigned);
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
    cudaError_t e = cudaFuncSetAttribute(select_heads_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         (int)kHeadSmemLimit);
    if (e != cudaSuccess) return e;
    return launch_dependent(select_heads_kernel, dim3(n_planes), dim3(kHeadThreads), smem, s, a);
}

}  // namespace deltas
