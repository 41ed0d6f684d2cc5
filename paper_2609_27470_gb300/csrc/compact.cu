// In-place, stream-order KV compaction (Alg. 1 "KV <- KV[I_sink u I_DeltaS u I_window]",
// applied to every full-attention layer; Sec. 3.3: survivors keep their original positions) and
// the per-chunk append to the caches (Alg. 1 Prefill).
//
// The gather row[j] <- row[retain_idx[j]] runs in place.  Because retain_idx is ascending with
// retain_idx[j] >= j, the only hazard is a destination row that is still to be read as the
// source of an earlier destination.  The work is cut into units (plane p, tile b of TB
// destination rows, starting at the tile of the first row that moves); a unit
//   1. stages the source rows of its tile in shared memory (TMA bulk copies, one per run of
//      consecutive sources),
//   2. publishes "tile b of plane p has been read" (release flag),
//   3. waits until every earlier tile whose destinations read rows of tile b has published
//      (the first such tile, need[b], comes from a prepass over retain_idx; the warp checks up to
//      32 flags at once),
//   4. writes its tile with one bulk store (the destination rows of a tile are contiguous).
// A unit publishes as soon as its own loads have landed, never after a wait, so no wait chains
// form across tiles.  Units are claimed through an atomic ticket in tile-major order, so a unit
// only waits for units that were claimed earlier by running CTAs whose loads complete without
// waiting on anything: no deadlock.
// Every wait is bounded (about one second); a wait that runs out records DELTAS_ERR_TIMEOUT,
// raises the abort flag and skips its writes.  Traffic is the algorithmic minimum: each moved row
// is read once and written once; rows that do not move are not touched.
#include <climits>

#include "internal.cuh"
#include "tc_ptx.cuh"

namespace deltas {
namespace {

using namespace tc;

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
    grid_dep_launch();                                 // the prepass may be scheduled now
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
    grid_dep_wait();                                   // the reset (and all earlier work) is done
    grid_dep_launch();
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


__device__ __forceinline__ int load_acquire(const int32_t* p) {
    int v;
    asm volatile("ld.acquire.gpu.global.b32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
    return v;
}

__device__ __forceinline__ void store_release(int32_t* p, int v) {
    asm volatile("st.release.gpu.global.b32 [%0], %1;" :: "l"(p), "r"(v) : "memory");
}


// Bulk (TMA) copies between global and shared memory: 16-byte aligned addresses, sizes in
// multiples of 16 bytes.
__device__ __forceinline__ void bulk_load(void* dst, const void* src, uint32_t bytes, uint64_t* bar) {
    asm volatile("cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];"
                 :: "r"(smem_u32(dst)), "l"(src), "r"(bytes), "r"(smem_u32(bar)) : "memory");
}
__device__ __forceinline__ void bulk_store(void* dst, const void* src, uint32_t bytes) {
    asm volatile("cp.async.bulk.global.shared::cta.bulk_group [%0], [%1], %2;"
                 :: "l"(dst), "r"(smem_u32(src)), "r"(bytes) : "memory");
}
__device__ __forceinline__ void fence_proxy_async() { asm volatile("fence.proxy.async;" ::: "memory"); }

// One warp per CTA (several CTAs per SM): claim a unit, load its moved source rows, publish, wait
// for the earlier readers of this tile, store.  For key / value planes the rows move by TMA bulk
// copies (one per run of consecutive sources, split at 32-row boundaries) into a shared-memory
// stage and back out in one bulk store; the 4-byte metadata rows go through registers.  A CTA
// never holds a claimed unit that it has not loaded and published while it waits on another one.
__global__ void __launch_bounds__(32)
compact_main_kernel(CompactArgs a)
{
    extern __shared__ uint4 stage_raw[];
    uint8_t* stage = reinterpret_cast<uint8_t*>(stage_raw);
    __shared__ uint64_t bar;

    grid_dep_wait();                                   // the prepass is done
    volatile int* abort_flag = &a.ctl->abort;
    if (*abort_flag) return;
    const int n = *a.n_retained;
    const int first = a.ctl->first;
    if (first >= n) return;                                        // nothing moves
    const int t0 = first / a.tile_rows;                            // tiles before t0 stay put
    const int n_tiles = (n + a.tile_rows - 1) / a.tile_rows;
    const int units = (n_tiles - t0) * a.n_planes;
    const int lane = threadIdx.x;
    if (lane == 0) { mbar_init(&bar, 1); fence_barrier_init(); }
    __syncwarp();

    uint32_t phase = 0;
    bool store_pending = false;                                    // lane 0's bulk store in flight
    bool load_pending = false;
    for (;;) {
        int u = 0;
        if (lane == 0) u = (*abort_flag) ? units : (int)atomicAdd(&a.ctl->ticket, 1u);
        u = __shfl_sync(0xffffffffu, u, 0);
        if (u >= units) break;
        const int b = t0 + u / a.n_planes, p = u % a.n_planes;
        int rb;
        char* base = plane_base(a, p, rb);
        const int j0 = b * a.tile_rows;
        const int j_end = min(j0 + a.tile_rows, n);
        const int js = max(j0, first);                             // rows before `first` stay
        const int nrows = j_end - js;
        const bool kv = rb >= 16;

        // ---- load the sources
        bool ok = true;
        if (kv) {
            if (lane == 0) {
                if (store_pending) bulk_wait_read0();              // the stage is free again
                mbar_arrive_expect_tx(&bar, (uint32_t)nrows * rb);
            }
            __syncwarp();
            for (int c0 = js; c0 < j_end; c0 += 32) {
                const int r = c0 + lane;
                const bool in = r < j_end;
                const int src = in ? a.retain_idx[r] : 0;
                int prev = __shfl_up_sync(0xffffffffu, src, 1);
                const bool start = in && (lane == 0 || src != prev + 1);
                const unsigned starts = __ballot_sync(0xffffffffu, start);
                if (start) {
                    const unsigned above = starts & ~((2u << lane) - 1u);   // later starts in this chunk
                    const int stop = above ? c0 + __ffs(above) - 1 : min(c0 + 32, j_end);
                    bulk_load(stage + (size_t)(r - j0) * rb, base + (size_t)src * rb, (uint32_t)(stop - r) * rb, &bar);
                }
            }
            load_pending = true;
            ok = mbar_wait_or_abort(&bar, phase, kWaitBudgetNs, abort_flag);
            ok = __all_sync(0xffffffffu, ok) != 0;
            if (ok) { phase ^= 1; load_pending = false; }
        } else {                                                   // 4-byte rows via the stage
            if (lane == 0 && store_pending) bulk_wait_read0();
            __syncwarp();
            int* st = reinterpret_cast<int*>(stage);
            for (int r = js + lane; r < j_end; r += 32) st[r - j0] = reinterpret_cast<const int*>(base)[a.retain_idx[r]];
            __syncwarp();
        }
        if (!ok) {
            if (lane == 0) { atomicExch(&a.ctl->abort, 1); record_status(a.status, DELTAS_ERR_TIMEOUT, u); }
            break;
        }

        // ---- publish, then wait (warp-parallel) for the earlier tiles that read this tile's rows
        if (lane == 0) {
            fence_proxy_async();
            __threadfence();
            store_release(a.flags + (size_t)p * a.max_tiles + b, 1);
        }
        const int first_reader = a.need[b];
        const uint64_t t_start = global_ns();
        for (int bb = first_reader; bb < b && ok; bb += 32) {
            const int mine = bb + lane;
            const int32_t* f = a.flags + (size_t)p * a.max_tiles + mine;
            for (;;) {
                const bool ready = (mine >= b) || load_acquire(f) != 0;
                if (__all_sync(0xffffffffu, ready)) break;
                if (*abort_flag || global_ns() - t_start > kWaitBudgetNs) { ok = false; break; }
                __nanosleep(32);
            }
        }
        if (!ok) {
            if (lane == 0) { atomicExch(&a.ctl->abort, 1); record_status(a.status, DELTAS_ERR_TIMEOUT, u); }
            break;
        }

        // ---- store the tile (destination rows of a tile are contiguous)
        if (kv) {
            if (lane == 0) {
                fence_proxy_async();
                bulk_store(base + (size_t)js * rb, stage + (size_t)(js - j0) * rb, (uint32_t)nrows * rb);
                bulk_commit();
                store_pending = true;
            }
        } else {
            const int* st = reinterpret_cast<const int*>(stage);
            for (int r = js + lane; r < j_end; r += 32) reinterpret_cast<int*>(base)[r] = st[r - j0];
            __syncwarp();                                          // the stage is rewritten next
        }
    }
    if (lane == 0) {
        bulk_wait0();                                              // stores complete before exit
        if (load_pending) mbar_wait(&bar, phase, kWaitBudgetNs);   // abort path: loads land first
    }
    __syncwarp();
}

// Append: block b copies kAppendVecs 16-byte vectors of one plane (plane b / blocks_per_plane),
// each thread kAppendUnroll of them with the loads issued before the stores; the last blocks also
// write the chunk id and positions of the new rows.
constexpr int kAppendThreads = 256;
constexpr int kAppendUnroll = 4;
constexpr int kAppendVecs = kAppendThreads * kAppendUnroll;

__global__ void __launch_bounds__(kAppendThreads)
append_kv_kernel(char* k_cache, char* v_cache, int n_kv_planes, int capacity, int row_bytes, int cache_len,
                 const char* k_new, const char* v_new, int n_new, int32_t* tok_chunk, int32_t* tok_pos,
                 int chunk_id, int first_pos, int blocks_per_plane)
{
    const int b = blockIdx.x;
    const int n_copy_blocks = 2 * n_kv_planes * blocks_per_plane;
    if (b >= n_copy_blocks) {                                  // metadata of the new rows
        for (int i = (b - n_copy_blocks) * kAppendThreads + threadIdx.x; i < n_new;
             i += (gridDim.x - n_copy_blocks) * kAppendThreads) {
            tok_chunk[cache_len + i] = chunk_id;
            tok_pos[cache_len + i] = first_pos + i;
        }
        return;
    }
    const int pp = b / blocks_per_plane, chunk = b - pp * blocks_per_plane;
    const bool is_v = pp >= n_kv_planes;
    const size_t p = is_v ? pp - n_kv_planes : pp;
    const int vec_per_plane = (int)((size_t)n_new * row_bytes / 16);
    const uint4* src = reinterpret_cast<const uint4*>((is_v ? v_new : k_new) + p * (size_t)n_new * row_bytes);
    uint4* dst = reinterpret_cast<uint4*>((is_v ? v_cache : k_cache) + (p * (size_t)capacity + cache_len) * row_bytes);
    const int e0 = chunk * kAppendVecs + threadIdx.x;
    uint4 v[kAppendUnroll];
#pragma unroll
    for (int u = 0; u < kAppendUnroll; ++u) {
        const int e = e0 + u * kAppendThreads;
        if (e < vec_per_plane) v[u] = __ldcs(src + e);
    }
#pragma unroll
    for (int u = 0; u < kAppendUnroll; ++u) {
        const int e = e0 + u * kAppendThreads;
        if (e < vec_per_plane) dst[e] = v[u];
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
    // the prepass and the moves start while their predecessor finishes (each waits for it before
    // reading or writing anything); the flag reset above is not overlapped: it writes the
    // workspace that the preceding call may still be using
    e = launch_dependent(compact_need_kernel, dim3(min(4 * sms, (cache_len + 255) / 256)), dim3(256), 0, s, a);
    if (e != cudaSuccess) return e;

    const int smem = a.tile_rows * a.row_bytes;
    int per_sm = 0;
    e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, compact_main_kernel, 32, smem);
    if (e != cudaSuccess) return e;
    if (per_sm < 1) per_sm = 1;
    const int max_units = a.max_tiles * a.n_planes;
    const int grid = max(1, min(max_units, per_sm * sms));
    return launch_dependent(compact_main_kernel, dim3(grid), dim3(32), (size_t)smem, s, a);
}

cudaError_t launch_append_kv(const KvPlanes& kv, int cache_len, const void* k_new, const void* v_new,
                             int n_new, int chunk_id, int first_pos, cudaStream_t s)
{
    if (n_new <= 0) return cudaSuccess;
    const int rb = kv.D * elt_bytes(kv.dtype);
    const size_t vec_per_plane = (size_t)n_new * rb / 16;
    if (vec_per_plane > (size_t)INT_MAX / 2) return cudaErrorInvalidValue;
    const int blocks_per_plane = (int)((vec_per_plane + kAppendVecs - 1) / kAppendVecs);
    const long long copy_blocks = 2ll * kv.Lf * kv.Hkv * blocks_per_plane;
    const int meta_blocks = (n_new + kAppendThreads - 1) / kAppendThreads;
    if (copy_blocks + meta_blocks > INT_MAX) return cudaErrorInvalidValue;
    append_kv_kernel<<<(int)(copy_blocks + meta_blocks), kAppendThreads, 0, s>>>(
        static_cast<char*>(kv.k_cache), static_cast<char*>(kv.v_cache), kv.Lf * kv.Hkv, kv.capacity, rb, cache_len,
        static_cast<const char*>(k_new), static_cast<const char*>(v_new), n_new, kv.tok_chunk, kv.tok_pos, chunk_id,
        first_pos, blocks_per_plane);
    return cudaGetLastError();
}

}  // namespace deltas
