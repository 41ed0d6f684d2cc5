// In-place, stream-order KV compaction (Alg. 1 "KV <- KV[I_sink u I_DeltaS u I_window]",
// applied to every full-attention layer; Sec. 3.3: survivors keep their original positions) and
// the per-chunk append to the caches (Alg. 1 Prefill).  With a token signal ranked per KV head
// (Sec. 4.3) every (layer, head) plane has its own retain list and its own metadata rows; the
// same kernels then gather each plane by its list (one `need` table and first row per list).
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
// Every wait is bounded (about one second, or the workspace's budget); a wait that runs out
// records DELTAS_ERR_TIMEOUT, raises the abort flag and skips its writes.  Traffic is the algorithmic minimum: each moved row
// is read once and written once; rows that do not move are not touched.
#include <algorithm>
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
    int first_min;         // first destination row that moves, over all lists (INT_MAX: none)
};

struct CompactArgs {
    char* k_cache;
    char* v_cache;
    char* meta[3];         // 4-byte metadata arrays: tok_chunk, tok_pos, tok_score (per-head only)
    int n_kv_planes;       // Lf * Hkv planes in each of K and V
    int n_lists;           // 1: one list moves every plane; n_kv_planes: one list per (layer, head)
    int list_stride;       // elements between two lists of retain_idx
    int n_meta;            // metadata arrays: 2 (shared list) or 3 (per head)
    int capacity;
    int row_bytes;         // D * element size (multiple of 16)
    int tile_rows;         // TB
    int n_planes;          // 2 * n_kv_planes (K and V); metadata moves with the K planes
    int cache_len;
    int max_tiles;         // ceil(cache_len / TB)
    const int32_t* retain_idx;
    const int32_t* n_retained;
    CompactCtl* ctl;
    int32_t* first;        // [n_lists] first destination row that moves (INT_MAX: none)
    int32_t* need;         // [n_lists][max_tiles]
    int32_t* flags;        // [n_planes][max_tiles]
    int32_t* status;
};

__host__ __device__ inline size_t align256(size_t x) { return (x + 255) & ~size_t(255); }

// Plane p of the unit order: K planes, then V planes.  Returns its base and the retain list that
// moves it.  The metadata rows (4 bytes per slot) ride with the K plane that owns them: with one
// shared list K plane 0 moves tok_chunk and tok_pos, with one list per (layer, head) K plane p
// moves row p of tok_chunk, tok_pos and tok_score.
__device__ __forceinline__ char* plane_base(const CompactArgs& a, int p, int& list, bool& owns_meta) {
    const bool shared_list = a.n_lists == 1;
    if (p < a.n_kv_planes) {
        list = shared_list ? 0 : p;
        owns_meta = shared_list ? p == 0 : true;
        return a.k_cache + (size_t)p * a.capacity * a.row_bytes;
    }
    p -= a.n_kv_planes;
    list = shared_list ? 0 : p;
    owns_meta = false;
    return a.v_cache + (size_t)p * a.capacity * a.row_bytes;
}

__global__ void compact_init_kernel(CompactArgs a) {
    grid_dep_launch();                                 // the prepass may be scheduled now
    grid_dep_wait();                                   // the previous call (which may share the
                                                       // workspace) is done before the reset
    const int total = a.n_planes * a.max_tiles;
    for (int e = blockIdx.x * blockDim.x + threadIdx.x; e < total + a.n_lists; e += gridDim.x * blockDim.x) {
        if (e < total) a.flags[e] = 0;
        else a.first[e - total] = INT_MAX;
    }
    if (blockIdx.x == 0 && threadIdx.x == 0) { a.ctl->ticket = 0; a.ctl->abort = 0; a.ctl->first_min = INT_MAX; }
}

// Validates every retain list and records, per list and source tile, the first destination tile
// that reads from it (itself if none does), and the list's first destination row that moves.  A
// list is ascending, so the rows reading one source tile are consecutive: the first of them
// writes need[] for its source tile and for the unread tiles before it, each tile exactly once.
// Rows with retain_idx[j] == j form a prefix (a moved row pushes every later source further on).
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
    const long long total = (long long)n * a.n_lists;
    for (long long e = blockIdx.x * (long long)blockDim.x + threadIdx.x; e < total;
         e += (long long)gridDim.x * blockDim.x) {
        const int l = (int)(e / n), j = (int)(e - (long long)l * n);
        const int32_t* ri = a.retain_idx + (size_t)l * a.list_stride;
        int32_t* need = a.need + (size_t)l * a.max_tiles;
        const int src = ri[j];
        const int prev = j > 0 ? ri[j - 1] : -1;
        const bool ok = src >= j && src < a.cache_len && src > prev;
        if (!ok) {
            atomicExch(&a.ctl->abort, 1);
            record_status(a.status, DELTAS_ERR_DEVICE_INDEX, j);
            continue;
        }
        const int ts = src / a.tile_rows, td = j / a.tile_rows;
        const int tp = prev < 0 ? -1 : prev / a.tile_rows;
        if (ts != tp) {
            for (int t = tp + 1; t < ts; ++t) need[t] = t;          // unread tiles
            need[ts] = td;
        }
        if (j == n - 1)
            for (int t = ts + 1; t < a.max_tiles; ++t) need[t] = t;
        if (src != j && prev == j - 1) {                           // unique: the list's first moved row
            a.first[l] = j;
            atomicMin(&a.ctl->first_min, j);
        }
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
// for the earlier readers of this tile, store.  The rows move by TMA bulk copies (one per run of
// consecutive sources, split at 32-row boundaries) into a shared-memory stage and back out in one
// bulk store; a K unit that owns metadata also gathers those words (plain loads into a second
// stage) before it publishes and writes them after its wait, so they follow the same hazard rule
// as its rows.  A CTA never holds a claimed unit that it has not loaded and published while it
// waits on another one.
__global__ void __launch_bounds__(32)
compact_main_kernel(CompactArgs a)
{
    extern __shared__ uint4 stage_raw[];
    uint8_t* stage = reinterpret_cast<uint8_t*>(stage_raw);
    int32_t* mstage = reinterpret_cast<int32_t*>(stage + (size_t)a.tile_rows * a.row_bytes);   // [n_meta][TB]
    __shared__ uint64_t bar;

    grid_dep_wait();                                   // the prepass is done
    volatile int* abort_flag = &a.ctl->abort;
    const uint64_t budget = wait_budget_ns(a.status);  // the drain below keeps kWaitBudgetNs
    if (*abort_flag) return;
    const int n = *a.n_retained;
    const int first_min = a.ctl->first_min;
    if (first_min >= n) return;                                    // nothing moves
    const int t0 = first_min / a.tile_rows;                        // tiles before t0 stay put
    const int n_tiles = (n + a.tile_rows - 1) / a.tile_rows;
    const int units = (n_tiles - t0) * a.n_planes;
    const int lane = threadIdx.x;
    const int rb = a.row_bytes;
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
        int list;
        bool owns_meta;
        char* base = plane_base(a, p, list, owns_meta);
        const int32_t* retain_idx = a.retain_idx + (size_t)list * a.list_stride;
        const int j0 = b * a.tile_rows;
        const int j_end = min(j0 + a.tile_rows, n);
        const int js = max(j0, a.first[list]);                     // rows before the list's first stay
        if (js >= j_end) continue;                                 // (no unit ever waits for such a tile)
        const int nrows = j_end - js;
        const size_t meta_off = (size_t)(a.n_lists == 1 ? 0 : list) * a.capacity;

        // ---- load the sources
        if (lane == 0) {
            if (store_pending) bulk_wait_read0();                  // the stage is free again
            mbar_arrive_expect_tx(&bar, (uint32_t)nrows * rb);
        }
        __syncwarp();
        for (int c0 = js; c0 < j_end; c0 += 32) {
            const int r = c0 + lane;
            const bool in = r < j_end;
            const int src = in ? retain_idx[r] : 0;
            int prev = __shfl_up_sync(0xffffffffu, src, 1);
            const bool start = in && (lane == 0 || src != prev + 1);
            const unsigned starts = __ballot_sync(0xffffffffu, start);
            if (start) {
                const unsigned above = starts & ~((2u << lane) - 1u);   // later starts in this chunk
                const int stop = above ? c0 + __ffs(above) - 1 : min(c0 + 32, j_end);
                bulk_load(stage + (size_t)(r - j0) * rb, base + (size_t)src * rb, (uint32_t)(stop - r) * rb, &bar);
            }
            if (owns_meta && in)
                for (int m = 0; m < a.n_meta; ++m)
                    mstage[m * a.tile_rows + (r - j0)] = reinterpret_cast<const int32_t*>(a.meta[m])[meta_off + src];
        }
        load_pending = true;
        bool ok = mbar_wait_or_abort(&bar, phase, budget, abort_flag);
        ok = __all_sync(0xffffffffu, ok) != 0;
        if (ok) { phase ^= 1; load_pending = false; }
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
        const int first_reader = a.need[(size_t)list * a.max_tiles + b];
        const uint64_t t_start = global_ns();
        for (int bb = first_reader; bb < b && ok; bb += 32) {
            const int mine = bb + lane;
            const int32_t* f = a.flags + (size_t)p * a.max_tiles + mine;
            for (;;) {
                const bool ready = (mine >= b) || load_acquire(f) != 0;
                if (__all_sync(0xffffffffu, ready)) break;
                if (*abort_flag || global_ns() - t_start > budget) { ok = false; break; }
                __nanosleep(32);
            }
        }
        if (!ok) {
            if (lane == 0) { atomicExch(&a.ctl->abort, 1); record_status(a.status, DELTAS_ERR_TIMEOUT, u); }
            break;
        }

        // ---- store the tile (destination rows of a tile are contiguous) and the metadata
        if (lane == 0) {
            fence_proxy_async();
            bulk_store(base + (size_t)js * rb, stage + (size_t)(js - j0) * rb, (uint32_t)nrows * rb);
            bulk_commit();
            store_pending = true;
        }
        if (owns_meta) {
            for (int r = js + lane; r < j_end; r += 32)
                for (int m = 0; m < a.n_meta; ++m)
                    reinterpret_cast<int32_t*>(a.meta[m])[meta_off + r] = mstage[m * a.tile_rows + (r - j0)];
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
    grid_dep_wait();                                   // earlier work on the caches is done
    grid_dep_launch();
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

// Append with a token signal (Sec. 4.3: key norm -||k||, value norm ||v||, per KV head): one
// warp per (plane, new row) copies the key and the value row into the caches (lane l moves the
// 16-byte vectors l, l + 32, ...), sums the squares of the signal's row in float32 (each lane its
// own elements, then a butterfly over the lanes), and writes the row's score -- a correctly
// rounded square root, negated for keys -- with the plane's chunk id and position.
constexpr int kAppendHeadsWarps = 8;

__device__ __forceinline__ float sum_squares16(const uint4& v, bool bf16) {
    const uint32_t w[4] = {v.x, v.y, v.z, v.w};
    float s = 0.f;
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        if (bf16) {
            const float lo = __uint_as_float(w[i] << 16), hi = __uint_as_float(w[i] & 0xffff0000u);
            s = fmaf(lo, lo, s);
            s = fmaf(hi, hi, s);
        } else {
            const float x = __uint_as_float(w[i]);
            s = fmaf(x, x, s);
        }
    }
    return s;
}

__global__ void __launch_bounds__(kAppendHeadsWarps * 32)
append_kv_heads_kernel(char* k_cache, char* v_cache, int n_kv_planes, int capacity, int row_bytes, int bf16,
                       int cache_len, const char* k_new, const char* v_new, int n_new, int32_t* tok_chunk,
                       int32_t* tok_pos, float* tok_score, int key_signal, int chunk_id, int first_pos)
{
    grid_dep_wait();                                   // earlier work on the caches is done
    grid_dep_launch();
    const long long row = (long long)blockIdx.x * kAppendHeadsWarps + (threadIdx.x >> 5);
    if (row >= (long long)n_kv_planes * n_new) return;
    const int lane = threadIdx.x & 31;
    const int p = (int)(row / n_new), i = (int)(row - (long long)p * n_new);
    const size_t src = ((size_t)p * n_new + i) * row_bytes;
    const size_t slot = (size_t)p * capacity + cache_len + i;
    const uint4* ks = reinterpret_cast<const uint4*>(k_new + src);
    const uint4* vs = reinterpret_cast<const uint4*>(v_new + src);
    uint4* kd = reinterpret_cast<uint4*>(k_cache + slot * row_bytes);
    uint4* vd = reinterpret_cast<uint4*>(v_cache + slot * row_bytes);
    const int nv = row_bytes / 16;
    float s = 0.f;
    for (int e = lane; e < nv; e += 32) {
        const uint4 kr = __ldcs(ks + e), vr = __ldcs(vs + e);
        kd[e] = kr;
        vd[e] = vr;
        s += sum_squares16(key_signal ? kr : vr, bf16 != 0);
    }
#pragma unroll
    for (int m = 16; m >= 1; m >>= 1) s += __shfl_xor_sync(0xffffffffu, s, m);
    if (lane == 0) {
        const float r = __fsqrt_rn(s);
        tok_score[slot] = key_signal ? -r : r;
        tok_chunk[slot] = chunk_id;
        tok_pos[slot] = first_pos + i;
    }
}

int tile_rows_for(int row_bytes) {
    int tb = kStageBytes / row_bytes;
    return tb < 1 ? 1 : (tb > 1024 ? 1024 : tb);
}

struct CompactWsLayout {
    size_t ctl, first, need, flags, total;
};

// per_head: one list per (layer, head) and three metadata arrays per plane.
CompactWsLayout compact_layout(const KvPlanes& kv, int cache_len, bool per_head) {
    const int rb = kv.D * elt_bytes(kv.dtype);
    const int tb = tile_rows_for(rb);
    const size_t max_tiles = (size_t)((cache_len + tb - 1) / tb);
    const size_t mt = max_tiles > 0 ? max_tiles : 1;
    const size_t n_kv = (size_t)kv.Lf * kv.Hkv;
    const size_t n_lists = per_head ? n_kv : 1;
    const size_t n_planes = 2 * n_kv;
    CompactWsLayout l;
    l.ctl = kStatusBytes;
    l.first = l.ctl + 256;
    l.need = l.first + align256(sizeof(int32_t) * n_lists);
    l.flags = l.need + align256(sizeof(int32_t) * n_lists * mt);
    l.total = l.flags + align256(sizeof(int32_t) * n_planes * mt);
    return l;
}

cudaError_t launch_compact(const KvPlanes& kv, bool per_head, const int32_t* retain_idx, int list_stride,
                           const int32_t* n_retained, int cache_len, void* ws, int32_t* status, cudaStream_t s)
{
    if (cache_len <= 0) return cudaSuccess;
    const CompactWsLayout l = compact_layout(kv, cache_len, per_head);
    char* w = static_cast<char*>(ws);
    CompactArgs a;
    a.k_cache = static_cast<char*>(kv.k_cache);
    a.v_cache = static_cast<char*>(kv.v_cache);
    a.meta[0] = reinterpret_cast<char*>(kv.tok_chunk);
    a.meta[1] = reinterpret_cast<char*>(kv.tok_pos);
    a.meta[2] = reinterpret_cast<char*>(kv.tok_score);
    a.n_kv_planes = kv.Lf * kv.Hkv;
    a.n_lists = per_head ? a.n_kv_planes : 1;
    a.list_stride = per_head ? list_stride : 0;
    a.n_meta = per_head ? 3 : 2;
    a.capacity = kv.capacity;
    a.row_bytes = kv.D * elt_bytes(kv.dtype);
    a.tile_rows = tile_rows_for(a.row_bytes);
    a.n_planes = 2 * a.n_kv_planes;
    a.cache_len = cache_len;
    a.max_tiles = (cache_len + a.tile_rows - 1) / a.tile_rows;
    a.retain_idx = retain_idx;
    a.n_retained = n_retained;
    a.ctl = reinterpret_cast<CompactCtl*>(w + l.ctl);
    a.first = reinterpret_cast<int32_t*>(w + l.first);
    a.need = reinterpret_cast<int32_t*>(w + l.need);
    a.flags = reinterpret_cast<int32_t*>(w + l.flags);
    a.status = status;

    const int sms = device_sm_count();
    const long long init_items = (long long)a.n_planes * a.max_tiles + a.n_lists;
    const int init_blocks = (int)std::min<long long>(4ll * sms, (init_items + 255) / 256 + 1);
    cudaError_t e = launch_dependent(compact_init_kernel, dim3(init_blocks), dim3(256), 0, s, a);
    if (e != cudaSuccess) return e;
    // the reset, the prepass and the moves start while their predecessor finishes (each waits for
    // it before reading or writing anything: the preceding call may share the workspace)
    const long long need_items = (long long)cache_len * a.n_lists;
    const int need_blocks = (int)std::min<long long>(4ll * sms, (need_items + 255) / 256);
    e = launch_dependent(compact_need_kernel, dim3(need_blocks), dim3(256), 0, s, a);
    if (e != cudaSuccess) return e;

    const int smem = a.tile_rows * (a.row_bytes + 4 * a.n_meta);
    int per_sm = 0;
    e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, compact_main_kernel, 32, smem);
    if (e != cudaSuccess) return e;
    if (per_sm < 1) per_sm = 1;
    const long long max_units = (long long)a.max_tiles * a.n_planes;
    const int grid = (int)std::max<long long>(1, std::min<long long>(max_units, (long long)per_sm * sms));
    return launch_dependent(compact_main_kernel, dim3(grid), dim3(32), (size_t)smem, s, a);
}

}  // namespace

size_t compact_workspace_bytes(const KvPlanes& kv, int cache_len) {
    return compact_layout(kv, cache_len, false).total;
}

size_t compact_heads_workspace_bytes(const KvPlanes& kv, int cache_len) {
    return compact_layout(kv, cache_len, true).total;
}

cudaError_t launch_compact_kv(const KvPlanes& kv, const int32_t* retain_idx, const int32_t* n_retained,
                              int cache_len, void* ws, int32_t* status, cudaStream_t s)
{
    return launch_compact(kv, false, retain_idx, 0, n_retained, cache_len, ws, status, s);
}

cudaError_t launch_compact_kv_heads(const KvPlanes& kv, const int32_t* retain_idx, int list_stride,
                                    const int32_t* n_retained, int cache_len, void* ws, int32_t* status,
                                    cudaStream_t s)
{
    return launch_compact(kv, true, retain_idx, list_stride, n_retained, cache_len, ws, status, s);
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
    // scheduled while the previous kernel finishes (it waits for it before touching memory)
    return launch_dependent(append_kv_kernel, dim3((int)(copy_blocks + meta_blocks)), dim3(kAppendThreads), 0, s,
                            static_cast<char*>(kv.k_cache), static_cast<char*>(kv.v_cache), kv.Lf * kv.Hkv,
                            kv.capacity, rb, cache_len, static_cast<const char*>(k_new),
                            static_cast<const char*>(v_new), n_new, kv.tok_chunk, kv.tok_pos, chunk_id, first_pos,
                            blocks_per_plane);
}

cudaError_t launch_append_kv_heads(const KvPlanes& kv, int signal, int cache_len, const void* k_new,
                                   const void* v_new, int n_new, int chunk_id, int first_pos, cudaStream_t s)
{
    if (n_new <= 0) return cudaSuccess;
    const int rb = kv.D * elt_bytes(kv.dtype);
    const long long rows = (long long)kv.Lf * kv.Hkv * n_new;
    const long long blocks = (rows + kAppendHeadsWarps - 1) / kAppendHeadsWarps;
    if (blocks > INT_MAX) return cudaErrorInvalidValue;
    return launch_dependent(append_kv_heads_kernel, dim3((int)blocks), dim3(kAppendHeadsWarps * 32), 0, s,
                            static_cast<char*>(kv.k_cache), static_cast<char*>(kv.v_cache), kv.Lf * kv.Hkv,
                            kv.capacity, rb, kv.dtype == DELTAS_BF16 ? 1 : 0, cache_len,
                            static_cast<const char*>(k_new), static_cast<const char*>(v_new), n_new, kv.tok_chunk,
                            kv.tok_pos, kv.tok_score, signal == DELTAS_SIGNAL_KEY_NORM ? 1 : 0, chunk_id, first_pos);
}

}  // namespace deltas
