// In-place, stream-order KV compaction (Alg. 1 "KV <- KV[I_sink u I_DeltaS u I_window]",
// applied to every full-attention layer; Sec. 3.3: survivors keep their original positions) and
// the per-chunk append to the caches (Alg. 1 Prefill).
//
// The gather row[j] <- row[retain_idx[j]] runs in place.  Because retain_idx is ascending with
// retain_idx[j] >= j, the only hazard is a destination row that is still to be read as the
// source of an earlier destination.  The work is cut into units (plane p, tile b of TB
// destination rows); a unit
//   1. stages the source rows of its tile in shared memory (16-byte cp.async loads),
//   2. publishes "tile b of plane p has been read" (release flag),
//   3. waits until every earlier tile whose destinations read rows of tile b has published
//      (the first such tile, need[b], comes from a prepass over retain_idx; one warp checks up to
//      32 flags at once),
//   4. writes its tile (16-byte stores; the destination rows of a tile are contiguous).
// A unit publishes as soon as its own loads have landed, never after a wait, so no wait chains
// form across tiles.  Units are claimed through an atomic ticket in tile-major order, so a unit
// only waits for units that were claimed earlier by running CTAs whose loads complete without
// waiting on anything: no deadlock.
// Every wait is bounded (about one second); a wait that runs out records DELTAS_ERR_TIMEOUT,
// raises the abort flag and skips its writes.  Traffic is the algorithmic minimum: each moved row
// is read once and written once; rows that do not move are not touched.
#include <climits>

#include "internal.cuh"

namespace deltas {
namespace {

constexpr int kCompactThreads = 256;
constexpr int kStageBytes = 32768;   // staged source rows of one unit

struct CompactCtl {
    unsigned ticket;
    int abort;
    int first;             // first destination row that moves (INT_MAX: none)
};

struct CompactArgs {
    char* k_cache;
    char* v_cache;
    char* tok_chunk;
    char* tok_pos;
    int n_kv_planes;       // Lf * Hkv planes in each of K and V
    int capacity;
    int row_bytes;         // D * element size (multiple of 16)
    int tile_rows;         // TB
    int n_planes;          // 2 * n_kv_planes + 2 (metadata)
    int cache_len;
    int max_tiles;         // ceil(cache_len / TB)
    const int32_t* retain_idx;
    const int32_t* n_retained;
    CompactCtl* ctl;
    int32_t* need;         // [max_tiles]
    int32_t* flags;        // [n_planes][max_tiles]
    int32_t* status;
};

__host__ __device__ inline size_t align256(size_t x) { return (x + 255) & ~size_t(255); }

__device__ __forceinline__ char* plane_base(const CompactArgs& a, int p, int& rb) {
    if (p < a.n_kv_planes) { rb = a.row_bytes; return a.k_cache + (size_t)p * a.capacity * a.row_bytes; }
    p -= a.n_kv_planes;
    if (p < a.n_kv_planes) { rb = a.row_bytes; return a.v_cache + (size_t)p * a.capacity * a.row_bytes; }
    rb = 4;
    return p == a.n_kv_planes ? a.tok_chunk : a.tok_pos;
}

__global__ void compact_init_kernel(CompactArgs a) {
    const int total = a.n_planes * a.max_tiles;
    for (int e = blockIdx.x * blockDim.x + threadIdx.x; e < total; e += gridDim.x * blockDim.x)
        a.flags[e] = 0;
    if (blockIdx.x == 0 && threadIdx.x == 0) { a.ctl->ticket = 0; a.ctl->abort = 0; a.ctl->first = INT_MAX; }
}

// Validates retain_idx and records, per source tile, the first destination tile that reads from
// it (itself if none does), and the first destination row that moves.  retain_idx is ascending,
// so the rows reading one source tile are consecutive: the first of them writes need[] for its
// source tile and for the unread tiles before it, each tile exactly once.  Rows with
// retain_idx[j] == j form a prefix (a moved row pushes every later source further on).
__global__ void compact_need_kernel(CompactArgs a) {
    const int n = *a.n_retained;
    if (n < 0 || n > a.cache_len) {
        if (blockIdx.x == 0 && threadIdx.x == 0) {
            a.ctl->abort = 1;
            record_status(a.status, DELTAS_ERR_DEVICE_INDEX, n);
        }
        return;
    }
    for (int j = blockIdx.x * blockDim.x + threadIdx.x; j < n; j += gridDim.x * blockDim.x) {
        const int src = a.retain_idx[j];
        const int prev = j > 0 ? a.retain_idx[j - 1] : -1;
        const bool ok = src >= j && src < a.cache_len && src > prev;
        if (!ok) {
            atomicExch(&a.ctl->abort, 1);
            record_status(a.status, DELTAS_ERR_DEVICE_INDEX, j);
            continue;
        }
        const int ts = src / a.tile_rows, td = j / a.tile_rows;
        const int tp = prev < 0 ? -1 : prev / a.tile_rows;
        if (ts != tp) {
            for (int t = tp + 1; t < ts; ++t) a.need[t] = t;        // unread tiles
            a.need[ts] = td;
        }
        if (j == n - 1)
            for (int t = ts + 1; t < a.max_tiles; ++t) a.need[t] = t;
        if (src != j && prev == j - 1) a.ctl->first = j;           // unique: the first moved row
    }
}

__device__ __forceinline__ bool warp_id_is_zero() { return (threadIdx.x >> 5) == 0; }

__device__ __forceinline__ int load_acquire(const int32_t* p) {
    int v;
    asm volatile("ld.acquire.gpu.global.b32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
    return v;
}

__device__ __forceinline__ void store_release(int32_t* p, int v) {
    asm volatile("st.release.gpu.global.b32 [%0], %1;" :: "l"(p), "r"(v) : "memory");
}

__device__ __forceinline__ void cp_async16(void* dst, const void* src) {
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16;"
                 :: "r"(static_cast<uint32_t>(__cvta_generic_to_shared(dst))), "l"(src) : "memory");
}
__device__ __forceinline__ void cp_async4(void* dst, const void* src) {
    asm volatile("cp.async.ca.shared.global [%0], [%1], 4;"
                 :: "r"(static_cast<uint32_t>(__cvta_generic_to_shared(dst))), "l"(src) : "memory");
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }
__device__ __forceinline__ void cp_async_wait_1() { asm volatile("cp.async.wait_group 1;" ::: "memory"); }
__device__ __forceinline__ void cp_async_wait_0() { asm volatile("cp.async.wait_group 0;" ::: "memory"); }

// Issues the asynchronous loads of one unit's moved source rows into a stage buffer.
__device__ __forceinline__ void compact_issue_loads(const CompactArgs& a, int b, int p, int n, uint8_t* stage) {
    int rb;
    const char* base = plane_base(a, p, rb);
    const int j0 = b * a.tile_rows;
    const int rows = min(a.tile_rows, n - j0);
    if (rb >= 16) {
        const int vpr = rb >> 4;
        const int nv = rows * vpr;
        for (int e = threadIdx.x; e < nv; e += kCompactThreads) {
            const int r = e / vpr, c = e - r * vpr;
            const int src = a.retain_idx[j0 + r];
            if (src != j0 + r) cp_async16(stage + 16 * e, base + (size_t)src * rb + 16 * c);
        }
    } else {
        for (int r = threadIdx.x; r < rows; r += kCompactThreads) {
            const int src = a.retain_idx[j0 + r];
            if (src != j0 + r) cp_async4(stage + 4 * r, base + (size_t)src * 4);
        }
    }
}

// One unit at a time per CTA (several CTAs per SM keep the memory system busy): claim, load the
// moved source rows, publish, wait for the earlier readers of this tile, store.  A CTA never holds
// a claimed unit that it has not loaded and published while it waits on another one.
__global__ void __launch_bounds__(kCompactThreads)
compact_main_kernel(CompactArgs a)
{
    extern __shared__ uint4 stage_raw[];
    uint8_t* stage = reinterpret_cast<uint8_t*>(stage_raw);
    __shared__ int s_unit[2];
    __shared__ int s_ok;

    volatile int* abort_flag = &a.ctl->abort;
    if (*abort_flag) return;
    const int n = *a.n_retained;
    const int first = a.ctl->first;
    if (first >= n) return;                                        // nothing moves
    const int t0 = first / a.tile_rows;                            // tiles before t0 stay put
    const int n_tiles = (n + a.tile_rows - 1) / a.tile_rows;
    const int units = (n_tiles - t0) * a.n_planes;
    const int tid = threadIdx.x, lane = tid & 31;

    for (;;) {
        if (tid == 0) s_unit[0] = (*abort_flag) ? units : (int)atomicAdd(&a.ctl->ticket, 1u);
        __syncthreads();
        const int cur = s_unit[0];
        if (cur >= units) break;
        const int b = t0 + cur / a.n_planes, p = cur % a.n_planes;
        compact_issue_loads(a, b, p, n, stage);
        cp_async_commit();
        cp_async_wait_0();
        __syncthreads();
        if (warp_id_is_zero()) {
            // publish, then wait (warp-parallel) for the earlier tiles that read this tile's rows
            if (lane == 0) {
                __threadfence();
                store_release(a.flags + (size_t)p * a.max_tiles + b, 1);
            }
            const int first_reader = a.need[b];
            int ok = 1;
            const uint64_t t_start = global_ns();
            for (int bb = first_reader; bb < b && ok; bb += 32) {
                const int mine = bb + lane;
                const int32_t* f = a.flags + (size_t)p * a.max_tiles + mine;
                for (;;) {
                    const bool ready = (mine >= b) || load_acquire(f) != 0;
                    if (__all_sync(0xffffffffu, ready)) break;
                    if (*abort_flag || global_ns() - t_start > kWaitBudgetNs) { ok = 0; break; }
                    __nanosleep(32);
                }
            }
            if (lane == 0) {
                if (!ok) {
                    atomicExch(&a.ctl->abort, 1);
                    record_status(a.status, DELTAS_ERR_TIMEOUT, b * a.n_planes + p);
                }
                s_ok = ok;
            }
        }
        __syncthreads();
        if (!s_ok) break;
        {   // write the tile (destination rows of a tile are contiguous)
            int rb;
            char* base = plane_base(a, p, rb);
            const int j0 = b * a.tile_rows;
            const int rows = min(a.tile_rows, n - j0);
            if (rb >= 16) {
                const int vpr = rb >> 4;
                const int nv = rows * vpr;
                uint4* dst = reinterpret_cast<uint4*>(base + (size_t)j0 * rb);
                for (int e = tid; e < nv; e += kCompactThreads) {
                    const int r = e / vpr;
                    if (a.retain_idx[j0 + r] != j0 + r) __stcs(dst + e, reinterpret_cast<const uint4*>(stage)[e]);
                }
            } else {
                for (int r = tid; r < rows; r += kCompactThreads)
                    if (a.retain_idx[j0 + r] != j0 + r)
                        reinterpret_cast<int*>(base)[j0 + r] = reinterpret_cast<const int*>(stage)[r];
            }
        }
        __syncthreads();                       // the stage is rewritten by the next unit
    }
}

__global__ void append_kv_kernel(char* k_cache, char* v_cache, int n_kv_planes, int capacity,
                                 int row_bytes, int cache_len, const char* k_new, const char* v_new,
                                 int n_new, int32_t* tok_chunk, int32_t* tok_pos, int chunk_id,
                                 int first_pos)
{
    const size_t vec_per_plane = (size_t)n_new * row_bytes / 16;
    const size_t total = 2 * (size_t)n_kv_planes * vec_per_plane;
    const size_t stride = (size_t)gridDim.x * blockDim.x;
    for (size_t e = (size_t)blockIdx.x * blockDim.x + threadIdx.x; e < total; e += stride) {
        const size_t pp = e / vec_per_plane, off = e - pp * vec_per_plane;
        const bool is_v = pp >= (size_t)n_kv_planes;
        const size_t p = is_v ? pp - n_kv_planes : pp;
        const uint4* src = reinterpret_cast<const uint4*>((is_v ? v_new : k_new) + p * (size_t)n_new * row_bytes);
        uint4* dst = reinterpret_cast<uint4*>((is_v ? v_cache : k_cache) +
                                              (p * (size_t)capacity + cache_len) * row_bytes);
        dst[off] = __ldcs(src + off);
    }
    for (size_t i = (size_t)blockIdx.x * blockDim.x + threadIdx.x; i < (size_t)n_new; i += stride) {
        tok_chunk[cache_len + i] = chunk_id;
        tok_pos[cache_len + i] = first_pos + (int)i;
    }
}

int tile_rows_for(int row_bytes) {
    int tb = kStageBytes / row_bytes;
    return tb < 1 ? 1 : (tb > 1024 ? 1024 : tb);
}

struct CompactWsLayout {
    size_t ctl, need, flags, total;
};

CompactWsLayout compact_layout(const KvPlanes& kv, int cache_len) {
    const int rb = kv.D * elt_bytes(kv.dtype);
    const int tb = tile_rows_for(rb);
    const size_t max_tiles = (size_t)((cache_len + tb - 1) / tb);
    const size_t n_planes = 2 * (size_t)kv.Lf * kv.Hkv + 2;
    CompactWsLayout l;
    l.ctl = kStatusBytes;
    l.need = l.ctl + 256;
    l.flags = l.need + align256(sizeof(int32_t) * (max_tiles > 0 ? max_tiles : 1));
    l.total = l.flags + align256(sizeof(int32_t) * n_planes * (max_tiles > 0 ? max_tiles : 1));
    return l;
}

}  // namespace

size_t compact_workspace_bytes(const KvPlanes& kv, int cache_len) {
    return compact_layout(kv, cache_len).total;
}

cudaError_t launch_compact_kv(const KvPlanes& kv, const int32_t* retain_idx, const int32_t* n_retained,
                              int cache_len, void* ws, int32_t* status, cudaStream_t s)
{
    if (cache_len <= 0) return cudaSuccess;
    const CompactWsLayout l = compact_layout(kv, cache_len);
    char* w = static_cast<char*>(ws);
    CompactArgs a;
    a.k_cache = static_cast<char*>(kv.k_cache);
    a.v_cache = static_cast<char*>(kv.v_cache);
    a.tok_chunk = reinterpret_cast<char*>(kv.tok_chunk);
    a.tok_pos = reinterpret_cast<char*>(kv.tok_pos);
    a.n_kv_planes = kv.Lf * kv.Hkv;
    a.capacity = kv.capacity;
    a.row_bytes = kv.D * elt_bytes(kv.dtype);
    a.tile_rows = tile_rows_for(a.row_bytes);
    a.n_planes = 2 * a.n_kv_planes + 2;
    a.cache_len = cache_len;
    a.max_tiles = (cache_len + a.tile_rows - 1) / a.tile_rows;
    a.retain_idx = retain_idx;
    a.n_retained = n_retained;
    a.ctl = reinterpret_cast<CompactCtl*>(w + l.ctl);
    a.need = reinterpret_cast<int32_t*>(w + l.need);
    a.flags = reinterpret_cast<int32_t*>(w + l.flags);
    a.status = status;

    const int sms = device_sm_count();
    const int init_blocks = min(4 * sms, (a.n_planes * a.max_tiles + 255) / 256 + 1);
    compact_init_kernel<<<init_blocks, 256, 0, s>>>(a);
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return e;
    compact_need_kernel<<<min(4 * sms, (cache_len + 255) / 256), 256, 0, s>>>(a);
    e = cudaGetLastError();
    if (e != cudaSuccess) return e;

    const int smem = a.tile_rows * a.row_bytes;
    int per_sm = 0;
    e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, compact_main_kernel, kCompactThreads, smem);
    if (e != cudaSuccess) return e;
    if (per_sm < 1) per_sm = 1;
    const int max_units = a.max_tiles * a.n_planes;
    const int grid = max(1, min(max_units, per_sm * sms));
    compact_main_kernel<<<grid, kCompactThreads, smem, s>>>(a);
    return cudaGetLastError();
}

cudaError_t launch_append_kv(const KvPlanes& kv, int cache_len, const void* k_new, const void* v_new,
                             int n_new, int chunk_id, int first_pos, cudaStream_t s)
{
    if (n_new <= 0) return cudaSuccess;
    const int rb = kv.D * elt_bytes(kv.dtype);
    const size_t total_vec = 2 * (size_t)kv.Lf * kv.Hkv * n_new * rb / 16;
    const int sms = device_sm_count();
    const size_t want = (total_vec + 255) / 256;
    const int blocks = (int)(want < (size_t)(8 * sms) ? (want > 0 ? want : 1) : (size_t)(8 * sms));
    append_kv_kernel<<<blocks, 256, 0, s>>>(static_cast<char*>(kv.k_cache), static_cast<char*>(kv.v_cache),
                                           kv.Lf * kv.Hkv, kv.capacity, rb, cache_len,
                                           static_cast<const char*>(k_new), static_cast<const char*>(v_new),
                                           n_new, kv.tok_chunk, kv.tok_pos, chunk_id, first_pos);
    return cudaGetLastError();
}

}  // namespace deltas
