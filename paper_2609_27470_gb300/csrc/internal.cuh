// Internal declarations shared by the library's kernels and its C-ABI layer.
#pragma once

#include <cuda_runtime.h>
#include <cuda_bf16.h>
#include <stdint.h>

#include "../../include/deltas.h"

namespace deltas {

// ---------------------------------------------------------------------------------------------
// Device status word: the first 16 bytes of every workspace.
//   word[0] = first recorded deltas_status, word[1] = detail, word[2] = bounded-wait budget in
//   nanoseconds (0: kWaitBudgetNs), word[3] reserved.
// ---------------------------------------------------------------------------------------------
constexpr size_t kStatusBytes = 256;   // status word padded so the rest stays 256-byte aligned

__device__ __forceinline__ void record_status(int32_t* status, int32_t code, int32_t detail) {
    if (status == nullptr) return;
    if (atomicCAS(status, 0, code) == 0) {
        atomicExch(status + 1, detail);
    }
}

__device__ __forceinline__ uint64_t global_ns() {
    uint64_t t;
    asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
    return t;
}

// Bounded-wait budget for every device-side spin (inter-CTA flags, mbarriers): about one second.
constexpr uint64_t kWaitBudgetNs = 1000000000ull;

// The budget of one call's waits: word 2 of its workspace header (nanoseconds, set by
// deltas_set_wait_budget), or kWaitBudgetNs when that word is zero.
__device__ __forceinline__ uint64_t wait_budget_ns(const int32_t* status) {
    const uint32_t v = status != nullptr ? reinterpret_cast<const volatile uint32_t*>(status)[2] : 0u;
    return v != 0u ? (uint64_t)v : kWaitBudgetNs;
}

__device__ __forceinline__ float to_f32(float x) { return x; }
__device__ __forceinline__ float to_f32(__nv_bfloat16 x) { return __bfloat162float(x); }
template <typename T> __device__ __forceinline__ T from_f32(float x);
template <> __device__ __forceinline__ float from_f32<float>(float x) { return x; }
template <> __device__ __forceinline__ __nv_bfloat16 from_f32<__nv_bfloat16>(float x) { return __float2bfloat16_rn(x); }

inline int elt_bytes(int32_t dtype) { return dtype == DELTAS_BF16 ? 2 : 4; }

// Programmatic dependent launch.  A kernel launched with launch_dependent() may be scheduled while
// the previous kernel of the stream is still running (it then overlaps that kernel's tail and its
// own launch latency); before it touches anything earlier work wrote it calls grid_dep_wait(),
// which returns once the previous kernel has completed and its writes are visible (hardware
// managed: no flag, no spin).  A kernel calls grid_dep_launch() to let its dependent be scheduled
// before it ends; the dependent's wait still covers all of it.
__device__ __forceinline__ void grid_dep_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }
__device__ __forceinline__ void grid_dep_launch() { asm volatile("griddepcontrol.launch_dependents;" ::: "memory"); }

template <typename... KArgs, typename... Args>
cudaError_t launch_dependent(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem, cudaStream_t s,
                             Args... args) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = grid;
    cfg.blockDim = block;
    cfg.dynamicSmemBytes = smem;
    cfg.stream = s;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, kernel, args...);
}

// ---------------------------------------------------------------------------------------------
// Launch arguments
// ---------------------------------------------------------------------------------------------
struct GdnArgs {
    int L, Hk, Hv, dk, dv, T, dtype;
    float q_scale;
    const void* q;
    const void* k;
    const void* v;
    const float* g;
    const float* beta;
    float* state;
    void* out;
    float* partials;
    float* wnorm;            // [L][Hv] sums over the chunk of beta_t ||v_t - alpha_t S_{t-1} k_t||, or null
    int32_t* status;
    uint8_t* scratch;        // workspace past the status word (the tensor-core path's WY factors)
    size_t scratch_bytes;
};

struct KvPlanes {
    int Lf, Hkv, D, dtype, capacity;
    void* k_cache;
    void* v_cache;
    int32_t* tok_chunk;      // [capacity], or [Lf][Hkv][capacity] with a per-head signal
    int32_t* tok_pos;
    float* tok_score = nullptr;   // [Lf][Hkv][capacity]: per-head token scores (Sec. 4.3 signals)
};

// A batch of row copies for one kernel: segment s moves `rows` rows of row_bytes bytes (16-byte
// aligned rows, row_bytes a multiple of 4), row r at src + r * stride to dst + r * stride.
struct CopySeg {
    const uint8_t* src;
    uint8_t* dst;
    uint64_t row_bytes;
    uint64_t stride;
    int64_t rows;
};
constexpr int kMaxCopySegs = 8;
struct CopyBatch {
    CopySeg seg[kMaxCopySegs];
    int n;
};

// Kernel launchers (return the launch error, cudaSuccess when enqueued).
cudaError_t launch_gdn_update_simt(const GdnArgs& a, cudaStream_t s);
bool gdn_tc_shape(const GdnArgs& a);        // d = 128, bfloat16, tokens > 0
bool gdn_tc_supported(const GdnArgs& a);    // ... and the tensor-core path can be launched
// workspace past the status word for the tensor-core path (with or without the read-out)
size_t gdn_tc_scratch_bytes(int L, int Hv, int dk, int dv, int dtype, int T, bool out);
cudaError_t launch_gdn_update_tc(const GdnArgs& a, cudaStream_t s);
cudaError_t launch_state_drift(int L, int Hv, int dv, int dk, const float* sb, const float* sa,
                               float* partials, cudaStream_t s);
cudaError_t launch_score_write_norms(int L, int Hv, const float* wnorm, int n_tokens, int chunk_id, float* scores,
                                     cudaStream_t s);
cudaError_t launch_score_chunks(int L, int Hv, const float* partials, int chunk_id, float* scores,
                                cudaStream_t s);
size_t select_workspace_bytes(int cache_len);
cudaError_t launch_select_retain(const deltas_policy& p, int cache_len, int num_chunks,
                                 const int32_t* tok_chunk, const float* scores, int32_t* retain_idx,
                                 int32_t* n_retained, uint8_t* mask, void* ws, int32_t* status,
                                 cudaStream_t s);
size_t compact_workspace_bytes(const KvPlanes& kv, int cache_len);
cudaError_t launch_compact_kv(const KvPlanes& kv, const int32_t* retain_idx, const int32_t* n_retained,
                              int cache_len, void* ws, int32_t* status, cudaStream_t s);
cudaError_t launch_copy_batch(const CopyBatch& b, cudaStream_t s);
// Per-head token signals (key norm, value norm; Sec. 4.3).
cudaError_t launch_append_kv_heads(const KvPlanes& kv, int signal, int cache_len, const void* k_new,
                                   const void* v_new, int n_new, int chunk_id, int first_pos, cudaStream_t s);
size_t select_heads_workspace_bytes(int n_planes, int cache_len);
cudaError_t launch_select_heads(const deltas_policy& p, int n_planes, int cache_len, int plane_stride,
                                const int32_t* tok_chunk, const float* tok_score, int32_t* retain_idx,
                                int32_t* n_retained, uint8_t* mask, void* ws, int32_t* status, cudaStream_t s);
size_t compact_heads_workspace_bytes(const KvPlanes& kv, int cache_len);
cudaError_t launch_compact_kv_heads(const KvPlanes& kv, const int32_t* retain_idx, int list_stride,
                                    const int32_t* n_retained, int cache_len, void* ws, int32_t* status,
                                    cudaStream_t s);
cudaError_t launch_append_kv(const KvPlanes& kv, int cache_len, const void* k_new, const void* v_new,
                             int n_new, int chunk_id, int first_pos, cudaStream_t s);

int device_sm_count();     // the device's SMs (cached per device)
int context_sm_count();    // the SMs the current context may use (<= device_sm_count())

}  // namespace deltas
