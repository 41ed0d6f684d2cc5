// Retain selection (Sec. 3.3; Alg. 1 eviction branch): a grid-wide run scan, a one-CTA decision,
// a grid-wide emit.
//
// Every token of a chunk carries its chunk's score, so candidates form runs: maximal stretches
// of consecutive slots with the same arrival chunk.  Inside a run the ranking key
// (score desc, slot asc) orders tokens by slot, and two runs never interleave in slot order, so
// the token-level rule "keep the best tokens" keeps a prefix of each run.  The kernel therefore
// works on runs (tens of them in a streaming cache, at most one per candidate slot in general):
//
//   A. runs (a grid-wide kernel): each block validates 1024 slots' chunk ids and writes its run
//      starts, their count and the min / max candidate chunk; the decision kernel (one 1024-thread
//      CTA) scans the counts and gathers the starts in slot order;
//   B. per run: length, temporal span floor((chunk - c_lo) * N / (c_hi - c_lo + 1)), 64-bit key
//      (total-order score bits << 32 | ~first_slot): larger key = better token;
//   C. per span: the run where the span's quota min(q, |span|) runs out -> kept1[run];
//   D. fill: the same over all runs' remainders (key re-based at the first unkept slot) with
//      target R - sum(kept1) -> kept[run].  Up to 512 runs (a streaming cache holds about one run
//      per cached chunk) are ranked directly in shared memory; more go through a token-weighted
//      radix select (8 passes of 8 bits, one warp scans each span's histogram) on workspace arrays;
//   E. output (a second, grid-wide kernel): every slot writes itself to retain_idx if it lies in
//      its run's kept prefix; sink and window slots are copied through.
// Nothing is sorted; the cost is a few passes over the slots plus 16 passes over the runs.
#include <algorithm>

#include "internal.cuh"

namespace deltas {
namespace {

constexpr int kSelThreads = 1024;
constexpr int kSelWarps = kSelThreads / 32;
constexpr int kMaxSpans = 32;

enum SpanMode : int { kNone = 0, kAll = 1, kSome = 2 };

// Select -> emit handoff, in the workspace's status area after the 16-byte status word.
struct SelCtl {
    int emit;           // 1: the eviction path ran and the emit kernel writes the outputs
    int n_runs;
};
constexpr size_t kSelCtlOffset = 64;

struct SelWs {          // workspace arrays, each [cache_len]
    int32_t* run_start;
    int32_t* run_chunk;
    int32_t* run_len;
    int32_t* run_span;
    int32_t* kept1;
    int32_t* kept;
    int32_t* out_off;
    uint64_t* run_key;
};

__host__ __device__ inline size_t align256(size_t x) { return (x + 255) & ~size_t(255); }

__host__ __device__ inline SelWs carve(void* ws, int cap) {
    char* p = static_cast<char*>(ws) + kStatusBytes;
    SelWs w;
    const size_t i32 = align256(sizeof(int32_t) * (size_t)(cap > 0 ? cap : 1));
    w.run_start = reinterpret_cast<int32_t*>(p); p += i32;
    w.run_chunk = reinterpret_cast<int32_t*>(p); p += i32;
    w.run_len = reinterpret_cast<int32_t*>(p); p += i32;
    w.run_span = reinterpret_cast<int32_t*>(p); p += i32;
    w.kept1 = reinterpret_cast<int32_t*>(p); p += i32;
    w.kept = reinterpret_cast<int32_t*>(p); p += i32;
    w.out_off = reinterpret_cast<int32_t*>(p); p += i32;
    w.run_key = reinterpret_cast<uint64_t*>(p);
    return w;
}

__device__ __forceinline__ uint32_t score_order_bits(float s) {
    const uint32_t b = __float_as_uint(s);
    return (b & 0x80000000u) ? ~b : (b | 0x80000000u);
}

// Exclusive block scan of one int per thread (1024 threads); *total receives the sum.
__device__ int block_exclusive_scan(int v, int* warp_sums, int* total) {
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    int x = v;
#pragma unroll
    for (int m = 1; m < 32; m <<= 1) {
        const int y = __shfl_up_sync(0xffffffffu, x, m);
        if (lane >= m) x += y;
    }
    if (lane == 31) warp_sums[warp] = x;
    __syncthreads();
    if (warp == 0) {
        int w = warp_sums[lane];
        int s = w;
#pragma unroll
        for (int m = 1; m < 32; m <<= 1) {
            const int y = __shfl_up_sync(0xffffffffu, s, m);
            if (lane >= m) s += y;
        }
        warp_sums[lane] = s - w;               // exclusive prefix of the warp totals
        if (lane == 31) *total = s;
    }
    __syncthreads();
    const int r = warp_sums[warp] + x - v;
    __syncthreads();                           // warp_sums may be reused right after
    return r;
}

// Token-weighted top selection per group.  For every group j with mode[j] == kSome, finds the
// key K*_j of the item at which the cumulative weight, in descending key order, first reaches
// target[j]; on return prefix[j] = K*_j and target[j] = weight to take from that item
// (1 <= target[j] <= its weight).  Keys are unique.  One warp scans each group's histogram.
__device__ void weighted_select(int n_items, const uint64_t* keys, const int32_t* weights,
                                const int32_t* groups, int G, uint64_t* prefix, int* target,
                                const int* mode, unsigned* hist)
{
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    for (int j = threadIdx.x; j < G; j += kSelThreads) prefix[j] = 0;
    for (int pass = 0; pass < 8; ++pass) {
        const int shift = 56 - 8 * pass;
        for (int e = threadIdx.x; e < G * 256; e += kSelThreads) hist[e] = 0;
        __syncthreads();
        for (int r = threadIdx.x; r < n_items; r += kSelThreads) {
            const int j = groups ? groups[r] : 0;
            if (mode[j] != kSome) continue;
            const int w = weights[r];
            if (w <= 0) continue;
            const uint64_t key = keys[r];
            if (pass > 0 && (key >> (shift + 8)) != (prefix[j] >> (shift + 8))) continue;
            atomicAdd(&hist[j * 256 + (int)((key >> shift) & 255u)], (unsigned)w);
        }
        __syncthreads();
        for (int j = warp; j < G; j += kSelWarps) {
            if (mode[j] != kSome) continue;
            // lane l holds digits 255-8l .. 248-8l (descending digit order across lanes)
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
            const unsigned t = (unsigned)target[j];
            const unsigned hit = __ballot_sync(0xffffffffu, incl >= t);
            const int src = __ffs(hit) - 1;                // first lane whose prefix reaches t
            if (lane == src) {
                unsigned cum = incl - local;
                int digit = 255 - 8 * lane;
                for (int e = 0; e < 8; ++e, --digit) {
                    const unsigned c = hj[digit];
                    if (cum + c >= t) break;
                    cum += c;
                }
                prefix[j] |= (uint64_t)digit << shift;
                target[j] = (int)(t - cum);
            }
        }
        __syncthreads();
    }
}

struct SelArgs {
    int M, n_s, n_w, N, T, n_chunks;
    const int32_t* tok_chunk;
    const float* scores;
    int32_t* retain_idx;
    int32_t* n_retained;
    uint8_t* mask;
    int32_t* status;
    SelCtl* ctl;
    SelWs ws;
};

constexpr int kSmallRuns = 512;   // runs held in shared memory and ranked directly


// ---- A. runs, grid-wide: block k scans slots [1024 k, 1024 k + 1024) (4 per thread, coalesced):
// validates their chunk ids, flags the run starts among the candidates [lo, hi), and writes its
// starts in slot order to run_chunk[1024 k ...] with its count, the min / max candidate chunk and
// the highest bad slot (or -1) in slot k of run_len / kept / out_off / kept1 (the decision kernel
// reads these before it reuses the arrays).
constexpr int kScanThreads = 256;
constexpr int kScanPer = 4;
constexpr int kScanSlots = kScanThreads * kScanPer;

__global__ void __launch_bounds__(kScanThreads)
select_runs_kernel(SelArgs a)
{
    __shared__ int s_wsum[kScanThreads / 32];
    __shared__ int s_min[kScanThreads / 32], s_max[kScanThreads / 32], s_bad[kScanThreads / 32];
    grid_dep_launch();                                 // the decision kernel may be scheduled now
    grid_dep_wait();                                   // the cache's chunk ids (and all earlier work)
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int T = a.T, lo = a.n_s, hi = T - a.n_w;
    const int b0 = blockIdx.x * kScanSlots;
    int c[kScanPer], p[kScanPer];
#pragma unroll
    for (int u = 0; u < kScanPer; ++u) {                  // slot b0 + u * 256 + tid
        const int i = b0 + u * kScanThreads + tid;
        c[u] = i < T ? a.tok_chunk[i] : 0;
        p[u] = (i < T && i > lo) ? a.tok_chunk[i - 1] : INT_MIN;
    }
    int cmin = INT_MAX, cmax = INT_MIN, bad = -1, flags = 0;
#pragma unroll
    for (int u = 0; u < kScanPer; ++u) {
        const int i = b0 + u * kScanThreads + tid;
        if (i >= T) continue;
        if (c[u] < 0 || c[u] >= a.n_chunks) bad = i;
        if (i >= lo && i < hi) {
            cmin = min(cmin, c[u]); cmax = max(cmax, c[u]);
            if (i == lo || c[u] != p[u]) flags |= 1 << u;
        }
    }
    // starts in slot order: group u of 256 slots before group u + 1; inside a group by thread
    int rank_base = 0;
    for (int u = 0; u < kScanPer; ++u) {
        const bool f = (flags >> u) & 1;
        const unsigned bal = __ballot_sync(0xffffffffu, f);
        if (lane == 0) s_wsum[warp] = __popc(bal);
        __syncthreads();
        int before = 0, total = 0;
        for (int w = 0; w < kScanThreads / 32; ++w) {
            const int v = s_wsum[w];
            before += w < warp ? v : 0;
            total += v;
        }
        if (f) a.ws.run_chunk[b0 + rank_base + before + __popc(bal & ((1u << lane) - 1u))] = b0 + u * kScanThreads + tid;
        rank_base += total;
        __syncthreads();
    }
#pragma unroll
    for (int m = 16; m >= 1; m >>= 1) {
        cmin = min(cmin, __shfl_xor_sync(0xffffffffu, cmin, m));
        cmax = max(cmax, __shfl_xor_sync(0xffffffffu, cmax, m));
        bad = max(bad, __shfl_xor_sync(0xffffffffu, bad, m));
    }
    if (lane == 0) { s_min[warp] = cmin; s_max[warp] = cmax; s_bad[warp] = bad; }
    __syncthreads();
    if (tid == 0) {
        for (int w = 1; w < kScanThreads / 32; ++w) {
            cmin = min(cmin, s_min[w]); cmax = max(cmax, s_max[w]); bad = max(bad, s_bad[w]);
        }
        a.ws.run_len[blockIdx.x] = rank_base;
        a.ws.kept[blockIdx.x] = cmin;
        a.ws.out_off[blockIdx.x] = cmax;
        a.ws.kept1[blockIdx.x] = bad;
    }
}

__global__ void __launch_bounds__(kSelThreads, 1)
select_retain_kernel(SelArgs a)
{
    __shared__ int warp_sums[32];
    __shared__ int s_total;
    __shared__ int s_bad;
    __shared__ int s_cmin[kSelWarps], s_cmax[kSelWarps];
    __shared__ int s_span_total[kMaxSpans];
    __shared__ int s_mode[kMaxSpans];
    __shared__ int s_target[kMaxSpans];
    __shared__ uint64_t s_prefix[kMaxSpans];
    __shared__ unsigned s_hist[kMaxSpans * 256];
    __shared__ int s_fill_mode[1], s_fill_target[1];
    __shared__ uint64_t s_fill_prefix[1];
    __shared__ uint64_t s_rkey[kSmallRuns];
    __shared__ int s_rstart[kSmallRuns], s_rlen[kSmallRuns], s_rspan[kSmallRuns], s_rkept[kSmallRuns],
        s_roff[kSmallRuns];

    grid_dep_wait();                                   // the run scan (and all earlier work) is done
    grid_dep_launch();
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int T = a.T;
    const int n_blocks = (T + kScanSlots - 1) / kScanSlots;
    // per-block results of the run scan (read before the arrays are reused below)
    int b_cnt = 0, b_min = INT_MAX, b_max = INT_MIN, b_bad = -1;
    for (int k = tid; k < n_blocks; k += kSelThreads) {   // n_blocks <= 1024 for T <= 1M slots
        b_cnt = a.ws.run_len[k]; b_min = a.ws.kept[k]; b_max = a.ws.out_off[k]; b_bad = a.ws.kept1[k];
    }
    if (tid == 0) { s_bad = -1; a.ctl->emit = 0; }
    __syncthreads();
    if (b_bad >= 0) atomicMax(&s_bad, b_bad);
    __syncthreads();
    if (s_bad >= 0) {
        if (tid == 0) { record_status(a.status, DELTAS_ERR_DEVICE_INDEX, s_bad); *a.n_retained = 0; }
        return;
    }
    if (T <= a.M) {                                    // keep everything
        for (int i = tid; i < T; i += kSelThreads) {
            a.retain_idx[i] = i;
            if (a.mask) a.mask[i] = 1;
        }
        if (tid == 0) *a.n_retained = T;
        return;
    }

    const int N = a.N < 1 ? 1 : a.N;
    const int hi = T - a.n_w;
    const int R = a.M - a.n_s - a.n_w;
    const int quota = R / N;

    // ---- A (gather). block run counts -> offsets; starts copied to r_start in slot order
    const int b_off = block_exclusive_scan(b_cnt, warp_sums, &s_total);
    const int n_runs = s_total;
    int cmin = b_min, cmax = b_max;
#pragma unroll
    for (int m = 16; m >= 1; m >>= 1) {
        cmin = min(cmin, __shfl_xor_sync(0xffffffffu, cmin, m));
        cmax = max(cmax, __shfl_xor_sync(0xffffffffu, cmax, m));
    }
    if (lane == 0) { s_cmin[warp] = cmin; s_cmax[warp] = cmax; }
    if (tid < kMaxSpans) s_span_total[tid] = 0;
    // the small path's pair sums, in the radix path's histogram space after the block counts and
    // offsets of the gather below
    int* s_above = reinterpret_cast<int*>(s_hist) + 2 * kSelThreads;
    int* s_above2 = s_above + kSmallRuns;
    static_assert(2 * kSelThreads + 2 * kSmallRuns <= kMaxSpans * 256, "histogram space");
    for (int r = tid; r < kSmallRuns; r += kSelThreads) { s_above[r] = 0; s_above2[r] = 0; }
    __syncthreads();
    const bool small = n_runs <= kSmallRuns;
    int c_lo = s_cmin[lane], c_hi = s_cmax[lane];            // (kSelWarps == 32)
#pragma unroll
    for (int m = 16; m >= 1; m >>= 1) {
        c_lo = min(c_lo, __shfl_xor_sync(0xffffffffu, c_lo, m));
        c_hi = max(c_hi, __shfl_xor_sync(0xffffffffu, c_hi, m));
    }
    const long long span_width = (long long)c_hi - c_lo + 1;
    int* r_start = small ? s_rstart : a.ws.run_start;
    int* r_len = small ? s_rlen : a.ws.run_len;
    int* r_span = small ? s_rspan : a.ws.run_span;
    uint64_t* r_key = small ? s_rkey : a.ws.run_key;
    {
        // block counts / offsets through shared memory (the radix path's histogram space, not yet
        // in use); warp w copies the starts of blocks w, w + 32, ...
        int* s_bcnt = reinterpret_cast<int*>(s_hist);
        int* s_boff = s_bcnt + kSelThreads;
        if (tid < n_blocks) { s_bcnt[tid] = b_cnt; s_boff[tid] = b_off; }
        __syncthreads();
        for (int k = warp; k < n_blocks; k += kSelWarps) {
            const int cnt = s_bcnt[k], off = s_boff[k];
            for (int i = lane; i < cnt; i += 32) r_start[off + i] = a.ws.run_chunk[k * kScanSlots + i];
        }
    }
    __syncthreads();
    // ---- B. per-run length, span and key (larger key = better: score desc, first slot asc)
    for (int r = tid; r < n_runs; r += kSelThreads) {
        const int st = r_start[r];
        const int end = (r + 1 < n_runs) ? r_start[r + 1] : hi;
        const int c = a.tok_chunk[st];
        const int span = (int)(((long long)(c - c_lo) * N) / span_width);
        r_len[r] = end - st;
        r_span[r] = span;
        r_key[r] = ((uint64_t)score_order_bits(a.scores[c]) << 32) | (uint64_t)(~(uint32_t)st);
        atomicAdd(&s_span_total[span], end - st);
    }
    __syncthreads();
    if (tid < N) {
        const int tot = s_span_total[tid];
        const int m = min(quota, tot);
        s_target[tid] = m;
        s_mode[tid] = (m == 0) ? kNone : (m == tot ? kAll : kSome);
    }
    __syncthreads();
    int granted = 0;
    for (int jj = 0; jj < N; ++jj) granted += s_target[jj];
    const int fill = R - granted;

    if (small) {
        // ---- C/D (at most 512 runs): a run keeps the part of its span quota (then of the fill)
        // that the runs ranked above it leave over.  The weight above run i is summed over all
        // pairs (i, r) by the whole CTA: thread t takes run i = t mod P (P = 32 or the next power
        // of two >= n_runs) and the t / P-th of 1024 / P slices of the runs r.
        const int P = n_runs <= 32 ? 32 : 1 << (32 - __clz(n_runs - 1));
        const int n_sl = kSelThreads / P;
        const int i = tid & (P - 1), sl = tid / P;
        const int per = (n_runs + n_sl - 1) / n_sl;
        const int r_lo = min(sl * per, n_runs), r_hi = min(r_lo + per, n_runs);
        if (i < n_runs) {
            const int j = s_rspan[i];
            const uint64_t key = s_rkey[i];
            int above = 0;
            for (int r = r_lo; r < r_hi; ++r)
                if (s_rspan[r] == j && s_rkey[r] > key) above += s_rlen[r];
            if (above) atomicAdd(&s_above[i], above);
        }
        __syncthreads();
        int k1 = 0, rem = 0;
        if (tid < n_runs) {
            const int len = s_rlen[tid];
            k1 = min(len, max(0, s_target[s_rspan[tid]] - s_above[tid]));
            rem = len - k1;
            s_rlen[tid] = rem;
            s_rkey[tid] = (s_rkey[tid] & 0xFFFFFFFF00000000ull) | (uint64_t)(~(uint32_t)(s_rstart[tid] + k1));
        }
        __syncthreads();
        if (fill > 0 && i < n_runs && s_rlen[i] > 0) {
            const uint64_t key2 = s_rkey[i];
            int above = 0;
            for (int r = r_lo; r < r_hi; ++r)
                if (s_rkey[r] > key2) above += s_rlen[r];
            if (above) atomicAdd(&s_above2[i], above);
        }
        __syncthreads();
        int kept = 0;
        if (tid < n_runs) {
            const int k2 = (fill > 0 && rem > 0) ? min(rem, max(0, fill - s_above2[tid])) : 0;
            kept = k1 + k2;
            s_rkept[tid] = kept;
        }
        const int off = block_exclusive_scan(kept, warp_sums, &s_total);
        if (tid < n_runs) s_roff[tid] = off;
        __syncthreads();
    } else {
        // ---- C. per-span quota by token-weighted radix selection
        weighted_select(n_runs, a.ws.run_key, a.ws.run_len, a.ws.run_span, N, s_prefix, s_target,
                        s_mode, s_hist);
        for (int r = tid; r < n_runs; r += kSelThreads) {
            const int j = a.ws.run_span[r];
            const int len = a.ws.run_len[r];
            int k1 = 0;
            if (s_mode[j] == kAll) k1 = len;
            else if (s_mode[j] == kSome) {
                const uint64_t key = a.ws.run_key[r];
                k1 = key > s_prefix[j] ? len : (key == s_prefix[j] ? s_target[j] : 0);
            }
            a.ws.kept1[r] = k1;
            a.ws.run_len[r] = len - k1;
            a.ws.run_key[r] = (a.ws.run_key[r] & 0xFFFFFFFF00000000ull) |
                              (uint64_t)(~(uint32_t)(a.ws.run_start[r] + k1));
        }
        if (tid == 0) {
            s_fill_target[0] = fill;
            s_fill_mode[0] = fill > 0 ? kSome : kNone;
        }
        __syncthreads();
        // ---- D. fill the unused capacity from the best remaining candidates
        weighted_select(n_runs, a.ws.run_key, a.ws.run_len, nullptr, 1, s_fill_prefix, s_fill_target,
                        s_fill_mode, s_hist);
        const int per = (n_runs + kSelThreads - 1) / kSelThreads;
        const int r_lo = min(tid * per, n_runs), r_hi = min(r_lo + per, n_runs);
        int my_kept = 0;
        for (int r = r_lo; r < r_hi; ++r) {
            const int remr = a.ws.run_len[r];
            int k2 = 0;
            if (s_fill_mode[0] == kSome && remr > 0) {
                const uint64_t key = a.ws.run_key[r];
                k2 = key > s_fill_prefix[0] ? remr : (key == s_fill_prefix[0] ? s_fill_target[0] : 0);
            }
            const int k = a.ws.kept1[r] + k2;
            a.ws.kept[r] = k;
            my_kept += k;
        }
        int off = block_exclusive_scan(my_kept, warp_sums, &s_total);
        for (int r = r_lo; r < r_hi; ++r) {
            a.ws.out_off[r] = off;
            off += a.ws.kept[r];
        }
        __syncthreads();
    }

    // ---- hand the runs to the emit kernel (E): the shared-memory arrays of the small path go to
    // the workspace, where the radix path keeps them already
    if (small) {
        for (int r = tid; r < n_runs; r += kSelThreads) {
            a.ws.run_start[r] = s_rstart[r];
            a.ws.kept[r] = s_rkept[r];
            a.ws.out_off[r] = s_roff[r];
        }
    }
    if (tid == 0) { a.ctl->n_runs = n_runs; a.ctl->emit = 1; }
    if (tid == 0) *a.n_retained = a.M;
}

// ---- E. every slot writes itself: a candidate slot goes to retain_idx if it lies in its run's
// kept prefix (its run found by binary search over the run starts); sink and window slots are
// copied through.  Grid-wide, one slot per thread.
constexpr int kEmitRuns = 2048;   // runs staged in shared memory by each emit block

__global__ void __launch_bounds__(256)
select_emit_kernel(SelArgs a)
{
    __shared__ int s_start[kEmitRuns], s_kept[kEmitRuns], s_off[kEmitRuns];
    grid_dep_wait();                                   // the decision is complete
    if (!a.ctl->emit) return;
    const int n_runs = a.ctl->n_runs;
    const int T = a.T, lo = a.n_s, hi = T - a.n_w;
    const bool staged = n_runs <= kEmitRuns;          // else the search runs on the workspace
    if (staged) {
        for (int r = threadIdx.x; r < n_runs; r += blockDim.x) {
            s_start[r] = a.ws.run_start[r]; s_kept[r] = a.ws.kept[r]; s_off[r] = a.ws.out_off[r];
        }
        __syncthreads();
    }
    const int* run_start = staged ? s_start : a.ws.run_start;
    const int* run_kept = staged ? s_kept : a.ws.kept;
    const int* run_off = staged ? s_off : a.ws.out_off;
    for (int i = blockIdx.x * blockDim.x + threadIdx.x; i < T; i += gridDim.x * blockDim.x) {
        if (i < lo) {
            a.retain_idx[i] = i;
            if (a.mask) a.mask[i] = 1;
        } else if (i >= hi) {
            a.retain_idx[a.M - a.n_w + (i - hi)] = i;
            if (a.mask) a.mask[i] = 1;
        } else {
            int l = 0, h = n_runs - 1;                     // last run with start <= i
            while (l < h) {
                const int m = (l + h + 1) >> 1;
                if (run_start[m] <= i) l = m; else h = m - 1;
            }
            const int pos = i - run_start[l];
            const bool keep = pos < run_kept[l];
            if (keep) a.retain_idx[a.n_s + run_off[l] + pos] = i;
            if (a.mask) a.mask[i] = keep ? 1 : 0;
        }
    }
}

}  // namespace

size_t select_workspace_bytes(int cache_len) {
    const size_t cap = (size_t)(cache_len > 0 ? cache_len : 1);
    return kStatusBytes + 7 * align256(sizeof(int32_t) * cap) + align256(sizeof(uint64_t) * cap);
}

cudaError_t launch_select_retain(const deltas_policy& p, int cache_len, int num_chunks,
                                 const int32_t* tok_chunk, const float* scores, int32_t* retain_idx,
                                 int32_t* n_retained, uint8_t* mask, void* ws, int32_t* status,
                                 cudaStream_t s)
{
    SelArgs a;
    a.M = p.budget_M; a.n_s = p.n_sink; a.n_w = p.n_window; a.N = p.n_buckets;
    a.T = cache_len; a.n_chunks = num_chunks;
    a.tok_chunk = tok_chunk; a.scores = scores; a.retain_idx = retain_idx;
    a.n_retained = n_retained; a.mask = mask; a.status = status;
    a.ctl = reinterpret_cast<SelCtl*>(static_cast<char*>(ws) + kSelCtlOffset);
    a.ws = carve(ws, cache_len);
    if (cache_len > 0) {
        const cudaError_t e0 = launch_dependent(select_runs_kernel, dim3((cache_len + kScanSlots - 1) / kScanSlots),
                                                dim3(kScanThreads), 0, s, a);
        if (e0 != cudaSuccess) return e0;
    }
    // the decision and the emission start while their predecessor finishes (each waits for it
    // before reading anything)
    cudaError_t e = launch_dependent(select_retain_kernel, dim3(1), dim3(kSelThreads), 0, s, a);
    if (e != cudaSuccess) return e;
    const int sms = device_sm_count();
    const int blocks = std::max(1, std::min((cache_len + 255) / 256, 2 * sms));
    return launch_dependent(select_emit_kernel, dim3(blocks), dim3(256), 0, s, a);
}

}  // namespace deltas

// -------------------------------------------------------------------------------------------------
// deltas_select_retain_static: the same selection with its scratch in this module's own device
// memory, for callers that may not allocate device memory at all (a runtime that owns every byte of
// HBM through its own pool or arena, or code running where cudaMalloc and friends are not allowed).
//
// The scratch is one file-scope array sized for DELTAS_SELECT_STATIC_MAX_CACHE_LEN slots.  Its
// address is looked up with cudaGetSymbolAddress on every call, with the caller's device current
// (the first call on a device loads the module there, so make it before any stream capture).  Every call on a device shares the array and
// finds it as the previous call left it: the status word at its head is the only part that has to
// start at zero, and it is cleared on the caller's stream before each launch; every other word the
// kernel reads was written earlier in the same launch.  Calls whose kernels can overlap on the GPU
// (different streams without ordering between them) race on the array.
// -------------------------------------------------------------------------------------------------
namespace {

constexpr size_t kStaticMaxSlots = DELTAS_SELECT_STATIC_MAX_CACHE_LEN;
// the layout carve() gives for kStaticMaxSlots slots: status word, 7 int32 arrays, 1 uint64 array
constexpr size_t kStaticScratchBytes =
    deltas::kStatusBytes + 7 * sizeof(int32_t) * kStaticMaxSlots + sizeof(uint64_t) * kStaticMaxSlots;
static_assert(kStaticScratchBytes % 256 == 0, "every scratch array must stay 256-byte aligned");

static __device__ __align__(256) unsigned char g_select_scratch[kStaticScratchBytes];

// The array's device address, looked up on every call: it belongs to the current context (a device
// reset or another context on the same device gives it another), and the lookup allocates nothing.
deltas_status static_scratch_for_current_device(void** out) {
    void* p = nullptr;
    if (cudaGetSymbolAddress(&p, g_select_scratch) != cudaSuccess || p == nullptr) return DELTAS_ERR_CUDA;
    *out = p;
    return DELTAS_OK;
}

}  // namespace

extern "C" deltas_status deltas_select_retain_static(const deltas_policy* policy, int32_t cache_len,
                                                     int32_t num_chunks, const int32_t* tok_chunk,
                                                     const float* chunk_scores, int32_t* retain_idx,
                                                     int32_t* n_retained, uint8_t* mask, void* stream)
{
    // the checks of deltas_select_retain, made here so that nothing is enqueued when one fails
    if (policy == nullptr || cache_len < 0 || num_chunks < 0) return DELTAS_ERR_INVALID_ARGUMENT;
    const deltas_policy& p = *policy;
    if (p.budget_M < 1 || p.n_sink < 0 || p.n_window < 0 || p.n_buckets < 0) return DELTAS_ERR_INVALID_ARGUMENT;
    if ((long long)p.budget_M < (long long)p.n_sink + p.n_window + 1) return DELTAS_ERR_INVALID_ARGUMENT;
    if (p.n_buckets > 32) return DELTAS_ERR_UNSUPPORTED;
    if (!retain_idx || !n_retained) return DELTAS_ERR_INVALID_ARGUMENT;
    if (cache_len > 0 && (!tok_chunk || !chunk_scores)) return DELTAS_ERR_INVALID_ARGUMENT;
    if ((size_t)cache_len > kStaticMaxSlots) return DELTAS_ERR_UNSUPPORTED;     // beyond the scratch

    void* scratch = nullptr;
    const deltas_status st = static_scratch_for_current_device(&scratch);
    if (st != DELTAS_OK) return st;
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    if (cudaMemsetAsync(scratch, 0, deltas::kStatusBytes, s) != cudaSuccess) return DELTAS_ERR_CUDA;
    const cudaError_t e = deltas::launch_select_retain(p, cache_len, num_chunks, tok_chunk, chunk_scores,
                                                       retain_idx, n_retained, mask, scratch,
                                                       static_cast<int32_t*>(scratch), s);
    return e == cudaSuccess ? DELTAS_OK : DELTAS_ERR_CUDA;
}
