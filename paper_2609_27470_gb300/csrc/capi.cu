// C-ABI entry points of libdeltas (declared and documented in include/deltas.h).
//
// This layer validates arguments on the host (nothing is enqueued when a check fails), carves the
// caller's workspace, and enqueues the kernels on the caller's stream.  It allocates nothing.
#include <algorithm>
#include <cstdint>
#include <cstring>
#include <mutex>

#include <cuda.h>

#include "internal.cuh"

namespace deltas {

// The SMs the current context may use: its SM resource (a green context's partition, the whole
// device for an ordinary context), else the device attribute.  Asked on every call: the answer
// belongs to the context, not to the device ordinal.  The driver calls come through the runtime's
// entry-point lookup (no link against libcuda).
int context_sm_count() {
    using GetCurrentFn = CUresult (*)(CUcontext*);
    using GetResourceFn = CUresult (*)(CUcontext, CUdevResource*, CUdevResourceType);
    static GetCurrentFn get_current = nullptr;
    static GetResourceFn get_resource = nullptr;
    static std::once_flag once;
    std::call_once(once, [] {
        cudaDriverEntryPointQueryResult q;
        void* p = nullptr;
        if (cudaGetDriverEntryPointByVersion("cuCtxGetCurrent", &p, 12000, cudaEnableDefault, &q) == cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            get_current = reinterpret_cast<GetCurrentFn>(p);
        p = nullptr;
        if (cudaGetDriverEntryPointByVersion("cuCtxGetDevResource", &p, 12040, cudaEnableDefault, &q) == cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            get_resource = reinterpret_cast<GetResourceFn>(p);
    });
    const int device = device_sm_count();
    if (get_current != nullptr && get_resource != nullptr) {
        CUcontext ctx = nullptr;
        if (get_current(&ctx) == CUDA_SUCCESS && ctx != nullptr) {
            CUdevResource r;
            std::memset(&r, 0, sizeof(r));
            if (get_resource(ctx, &r, CU_DEV_RESOURCE_TYPE_SM) == CUDA_SUCCESS && r.type == CU_DEV_RESOURCE_TYPE_SM &&
                r.sm.smCount > 0)
                return std::min((int)r.sm.smCount, device);
        }
    }
    return device;
}

int device_sm_count() {
    // cached per device: the attribute query is cheap but not free
    static int cached[64] = {0};
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0) return 1;
    if (dev < 64 && cached[dev] > 0) return cached[dev];
    int n = 0;
    if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || n < 1) n = 1;
    if (dev < 64) cached[dev] = n;
    return n;
}

}  // namespace deltas

using namespace deltas;

namespace {

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }
bool aligned256(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 255u) == 0; }
cudaStream_t as_stream(void* s) { return static_cast<cudaStream_t>(s); }

deltas_status check_gdn_desc(const deltas_gdn_desc* d) {
    if (d == nullptr) return DELTAS_ERR_INVALID_ARGUMENT;
    if (d->num_layers < 1 || d->num_k_heads < 1 || d->num_v_heads < 1) return DELTAS_ERR_INVALID_ARGUMENT;
    if (d->num_v_heads % d->num_k_heads != 0) return DELTAS_ERR_INVALID_ARGUMENT;
    if (d->key_dim < 1 || d->value_dim < 1) return DELTAS_ERR_INVALID_ARGUMENT;
    if (d->dtype != DELTAS_F32 && d->dtype != DELTAS_BF16) return DELTAS_ERR_INVALID_ARGUMENT;
    if (d->key_dim != d->value_dim) return DELTAS_ERR_UNSUPPORTED;
    if (d->key_dim != 16 && d->key_dim != 32 && d->key_dim != 64 && d->key_dim != 128) return DELTAS_ERR_UNSUPPORTED;
    if ((long long)d->num_layers * d->num_v_heads > (1ll << 30)) return DELTAS_ERR_UNSUPPORTED;
    return DELTAS_OK;
}

deltas_status check_workspace(const void* ws, size_t bytes, size_t need) {
    if (ws == nullptr || !aligned256(ws) || bytes < need) return DELTAS_ERR_WORKSPACE;
    return DELTAS_OK;
}

deltas_status check_kv_desc(const deltas_kv_desc* d) {
    if (d == nullptr) return DELTAS_ERR_INVALID_ARGUMENT;
    if (d->num_layers < 1 || d->num_kv_heads < 1 || d->head_dim < 1 || d->capacity < 0) return DELTAS_ERR_INVALID_ARGUMENT;
    if (d->dtype != DELTAS_F32 && d->dtype != DELTAS_BF16) return DELTAS_ERR_INVALID_ARGUMENT;
    if ((d->head_dim * elt_bytes(d->dtype)) % 16 != 0) return DELTAS_ERR_UNSUPPORTED;
    const long long rb = (long long)d->head_dim * elt_bytes(d->dtype);
    if (rb > 32768) return DELTAS_ERR_UNSUPPORTED;
    if ((long long)d->num_layers * d->num_kv_heads > (1ll << 20)) return DELTAS_ERR_UNSUPPORTED;
    return DELTAS_OK;
}

KvPlanes make_planes(const deltas_kv_desc* d, void* k, void* v, int32_t* tc, int32_t* tp) {
    KvPlanes p;
    p.Lf = d->num_layers; p.Hkv = d->num_kv_heads; p.D = d->head_dim; p.dtype = d->dtype;
    p.capacity = d->capacity; p.k_cache = k; p.v_cache = v; p.tok_chunk = tc; p.tok_pos = tp;
    return p;
}

deltas_status from_cuda(cudaError_t e) { return e == cudaSuccess ? DELTAS_OK : DELTAS_ERR_CUDA; }

}  // namespace

extern "C" {

const char* deltas_version(void) { return "deltas 0.1.0 sm_103a"; }

const char* deltas_status_string(int32_t s) {
    switch (s) {
        case DELTAS_OK: return "ok";
        case DELTAS_ERR_INVALID_ARGUMENT: return "invalid argument";
        case DELTAS_ERR_UNSUPPORTED: return "unsupported shape or dtype";
        case DELTAS_ERR_WORKSPACE: return "workspace missing, misaligned or too small";
        case DELTAS_ERR_CUDA: return "CUDA launch or runtime error";
        case DELTAS_ERR_TIMEOUT: return "device: bounded wait ran out";
        case DELTAS_ERR_DEVICE_INDEX: return "device: index out of range or out of order";
        default: return "unknown status";
    }
}

size_t deltas_gdn_chunk_update_workspace_size(const deltas_gdn_desc* desc, int32_t n_tokens) {
    if (desc == nullptr || n_tokens <= 0) return kStatusBytes;
    return kStatusBytes + gdn_tc_scratch_bytes(desc->num_layers, desc->num_v_heads, desc->key_dim,
                                               desc->value_dim, desc->dtype, n_tokens, false);
}

size_t deltas_gdn_chunk_update_readout_workspace_size(const deltas_gdn_desc* desc, int32_t n_tokens) {
    if (desc == nullptr || n_tokens <= 0) return kStatusBytes;
    return kStatusBytes + gdn_tc_scratch_bytes(desc->num_layers, desc->num_v_heads, desc->key_dim,
                                               desc->value_dim, desc->dtype, n_tokens, true);
}

namespace {

deltas_status gdn_update(const deltas_gdn_desc* desc, int32_t n_tokens, const void* q, const void* k,
                         const void* v, const float* g, const float* beta, float* state, void* out,
                         float* drift_partials, float* write_norms, void* workspace, size_t workspace_bytes,
                         void* stream)
{
    deltas_status st = check_gdn_desc(desc);
    if (st != DELTAS_OK) return st;
    if (n_tokens < 0) return DELTAS_ERR_INVALID_ARGUMENT;
    if (state == nullptr || !aligned16(state)) return DELTAS_ERR_INVALID_ARGUMENT;
    if (n_tokens > 0) {
        if (!k || !v || !g || !beta || !aligned16(k) || !aligned16(v)) return DELTAS_ERR_INVALID_ARGUMENT;
        if (out && (!q || !aligned16(q) || !aligned16(out))) return DELTAS_ERR_INVALID_ARGUMENT;
    }
    if (drift_partials && !aligned16(drift_partials)) return DELTAS_ERR_INVALID_ARGUMENT;
    if (write_norms && !aligned16(write_norms)) return DELTAS_ERR_INVALID_ARGUMENT;
    st = check_workspace(workspace, workspace_bytes,
                         out ? deltas_gdn_chunk_update_readout_workspace_size(desc, n_tokens)
                             : deltas_gdn_chunk_update_workspace_size(desc, n_tokens));
    if (st != DELTAS_OK) return st;
    GdnArgs a;
    a.L = desc->num_layers; a.Hk = desc->num_k_heads; a.Hv = desc->num_v_heads;
    a.dk = desc->key_dim; a.dv = desc->value_dim; a.T = n_tokens; a.dtype = desc->dtype;
    a.q_scale = desc->q_scale; a.q = q; a.k = k; a.v = v; a.g = g; a.beta = beta;
    a.state = state; a.out = out; a.partials = drift_partials; a.wnorm = write_norms;
    a.status = static_cast<int32_t*>(workspace);
    a.scratch = static_cast<uint8_t*>(workspace) + kStatusBytes;
    a.scratch_bytes = workspace_bytes - kStatusBytes;
    // d = 128 bfloat16 runs on the tensor cores or not at all: no silent fallback
    if (gdn_tc_shape(a)) {
        if (!gdn_tc_supported(a)) return DELTAS_ERR_UNSUPPORTED;
        return from_cuda(launch_gdn_update_tc(a, as_stream(stream)));
    }
    return from_cuda(launch_gdn_update_simt(a, as_stream(stream)));
}

}  // namespace

deltas_status deltas_gdn_chunk_update(const deltas_gdn_desc* desc, int32_t n_tokens,
                                      const void* q, const void* k, const void* v,
                                      const float* g, const float* beta,
                                      float* state, void* out, float* drift_partials,
                                      void* workspace, size_t workspace_bytes, void* stream)
{
    return gdn_update(desc, n_tokens, q, k, v, g, beta, state, out, drift_partials, nullptr, workspace,
                      workspace_bytes, stream);
}

deltas_status deltas_gdn_chunk_update_write_norms(const deltas_gdn_desc* desc, int32_t n_tokens,
                                                  const void* q, const void* k, const void* v,
                                                  const float* g, const float* beta,
                                                  float* state, void* out, float* drift_partials,
                                                  float* write_norms, void* workspace,
                                                  size_t workspace_bytes, void* stream)
{
    if (write_norms == nullptr) return DELTAS_ERR_INVALID_ARGUMENT;
    return gdn_update(desc, n_tokens, q, k, v, g, beta, state, out, drift_partials, write_norms, workspace,
                      workspace_bytes, stream);
}

size_t deltas_state_drift_workspace_size(const deltas_gdn_desc* desc) {
    (void)desc;
    return kStatusBytes;
}

deltas_status deltas_state_drift(const deltas_gdn_desc* desc, const float* s_before,
                                 const float* s_after, float* drift_partials,
                                 void* workspace, size_t workspace_bytes, void* stream)
{
    if (desc == nullptr) return DELTAS_ERR_INVALID_ARGUMENT;
    if (desc->num_layers < 1 || desc->num_v_heads < 1 || desc->key_dim < 1 || desc->value_dim < 1)
        return DELTAS_ERR_INVALID_ARGUMENT;
    if (((long long)desc->key_dim * desc->value_dim) % 4 != 0) return DELTAS_ERR_UNSUPPORTED;
    if ((long long)desc->key_dim * desc->value_dim > (1ll << 30)) return DELTAS_ERR_UNSUPPORTED;
    if (!s_before || !s_after || !drift_partials) return DELTAS_ERR_INVALID_ARGUMENT;
    if (!aligned16(s_before) || !aligned16(s_after)) return DELTAS_ERR_INVALID_ARGUMENT;
    deltas_status st = check_workspace(workspace, workspace_bytes, deltas_state_drift_workspace_size(desc));
    if (st != DELTAS_OK) return st;
    return from_cuda(launch_state_drift(desc->num_layers, desc->num_v_heads, desc->value_dim,
                                        desc->key_dim, s_before, s_after, drift_partials,
                                        as_stream(stream)));
}

deltas_status deltas_score_write_norms(int32_t num_layers, int32_t num_v_heads, const float* write_norms,
                                       int32_t n_tokens, int32_t chunk_id, float* chunk_scores, void* stream)
{
    if (num_layers < 1 || num_v_heads < 1 || n_tokens < 0 || chunk_id < 0) return DELTAS_ERR_INVALID_ARGUMENT;
    if ((long long)num_layers * num_v_heads > (1ll << 30)) return DELTAS_ERR_UNSUPPORTED;
    if (!write_norms || !chunk_scores) return DELTAS_ERR_INVALID_ARGUMENT;
    return from_cuda(launch_score_write_norms(num_layers, num_v_heads, write_norms, n_tokens, chunk_id,
                                              chunk_scores, as_stream(stream)));
}

deltas_status deltas_score_chunks(int32_t num_layers, int32_t num_v_heads,
                                  const float* drift_partials, int32_t chunk_id,
                                  float* chunk_scores, void* stream)
{
    if (num_layers < 1 || num_v_heads < 1 || chunk_id < 0) return DELTAS_ERR_INVALID_ARGUMENT;
    if (!drift_partials || !chunk_scores) return DELTAS_ERR_INVALID_ARGUMENT;
    return from_cuda(launch_score_chunks(num_layers, num_v_heads, drift_partials, chunk_id,
                                         chunk_scores, as_stream(stream)));
}

size_t deltas_select_retain_workspace_size(int32_t cache_len) {
    return select_workspace_bytes(cache_len);
}

deltas_status deltas_select_retain(const deltas_policy* policy, int32_t cache_len,
                                   int32_t num_chunks, const int32_t* tok_chunk,
                                   const float* chunk_scores, int32_t* retain_idx,
                                   int32_t* n_retained, uint8_t* mask,
                                   void* workspace, size_t workspace_bytes, void* stream)
{
    if (policy == nullptr || cache_len < 0 || num_chunks < 0) return DELTAS_ERR_INVALID_ARGUMENT;
    const deltas_policy& p = *policy;
    if (p.budget_M < 1 || p.n_sink < 0 || p.n_window < 0 || p.n_buckets < 0) return DELTAS_ERR_INVALID_ARGUMENT;
    if ((long long)p.budget_M < (long long)p.n_sink + p.n_window + 1) return DELTAS_ERR_INVALID_ARGUMENT;
    if (p.n_buckets > 32) return DELTAS_ERR_UNSUPPORTED;
    if (cache_len > DELTAS_SELECT_MAX_CACHE_LEN) return DELTAS_ERR_UNSUPPORTED;
    if (!retain_idx || !n_retained) return DELTAS_ERR_INVALID_ARGUMENT;
    if (cache_len > 0 && (!tok_chunk || !chunk_scores)) return DELTAS_ERR_INVALID_ARGUMENT;
    deltas_status st = check_workspace(workspace, workspace_bytes, deltas_select_retain_workspace_size(cache_len));
    if (st != DELTAS_OK) return st;
    return from_cuda(launch_select_retain(p, cache_len, num_chunks, tok_chunk, chunk_scores, retain_idx,
                                          n_retained, mask, workspace, static_cast<int32_t*>(workspace),
                                          as_stream(stream)));
}

size_t deltas_compact_kv_workspace_size(const deltas_kv_desc* desc, int32_t cache_len) {
    if (check_kv_desc(desc) != DELTAS_OK || cache_len < 0) return 0;
    KvPlanes kv = make_planes(desc, nullptr, nullptr, nullptr, nullptr);
    return compact_workspace_bytes(kv, cache_len);
}

deltas_status deltas_compact_kv(const deltas_kv_desc* desc, void* k_cache, void* v_cache,
                                int32_t* tok_chunk, int32_t* tok_pos,
                                const int32_t* retain_idx, const int32_t* n_retained,
                                int32_t cache_len, void* workspace, size_t workspace_bytes,
                                void* stream)
{
    deltas_status st = check_kv_desc(desc);
    if (st != DELTAS_OK) return st;
    if (cache_len < 0 || cache_len > desc->capacity) return DELTAS_ERR_INVALID_ARGUMENT;
    if (!k_cache || !v_cache || !tok_chunk || !tok_pos || !retain_idx || !n_retained) return DELTAS_ERR_INVALID_ARGUMENT;
    if (!aligned16(k_cache) || !aligned16(v_cache)) return DELTAS_ERR_INVALID_ARGUMENT;
    st = check_workspace(workspace, workspace_bytes, deltas_compact_kv_workspace_size(desc, cache_len));
    if (st != DELTAS_OK) return st;
    KvPlanes kv = make_planes(desc, k_cache, v_cache, tok_chunk, tok_pos);
    return from_cuda(launch_compact_kv(kv, retain_idx, n_retained, cache_len, workspace,
                                       static_cast<int32_t*>(workspace), as_stream(stream)));
}

deltas_status deltas_append_kv(const deltas_kv_desc* desc, void* k_cache, void* v_cache,
                               int32_t* tok_chunk, int32_t* tok_pos, int32_t cache_len,
                               const void* k_new, const void* v_new, int32_t n_new,
                               int32_t chunk_id, int32_t first_pos, void* stream)
{
    deltas_status st = check_kv_desc(desc);
    if (st != DELTAS_OK) return st;
    if (cache_len < 0 || n_new < 0 || (long long)cache_len + n_new > desc->capacity) return DELTAS_ERR_INVALID_ARGUMENT;
    if ((long long)first_pos + n_new > INT32_MAX || first_pos < 0) return DELTAS_ERR_INVALID_ARGUMENT;
    if (!k_cache || !v_cache || !tok_chunk || !tok_pos) return DELTAS_ERR_INVALID_ARGUMENT;
    if (n_new > 0 && (!k_new || !v_new || !aligned16(k_new) || !aligned16(v_new))) return DELTAS_ERR_INVALID_ARGUMENT;
    if (!aligned16(k_cache) || !aligned16(v_cache)) return DELTAS_ERR_INVALID_ARGUMENT;
    KvPlanes kv = make_planes(desc, k_cache, v_cache, tok_chunk, tok_pos);
    return from_cuda(launch_append_kv(kv, cache_len, k_new, v_new, n_new, chunk_id, first_pos,
                                      as_stream(stream)));
}

deltas_status deltas_append_kv_heads(const deltas_kv_desc* desc, int32_t signal, void* k_cache, void* v_cache,
                                     int32_t* tok_chunk, int32_t* tok_pos, float* tok_score, int32_t cache_len,
                                     const void* k_new, const void* v_new, int32_t n_new, int32_t chunk_id,
                                     int32_t first_pos, void* stream)
{
    deltas_status st = check_kv_desc(desc);
    if (st != DELTAS_OK) return st;
    if (signal != DELTAS_SIGNAL_KEY_NORM && signal != DELTAS_SIGNAL_VALUE_NORM) return DELTAS_ERR_INVALID_ARGUMENT;
    if (cache_len < 0 || n_new < 0 || (long long)cache_len + n_new > desc->capacity) return DELTAS_ERR_INVALID_ARGUMENT;
    if ((long long)first_pos + n_new > INT32_MAX || first_pos < 0) return DELTAS_ERR_INVALID_ARGUMENT;
    if (!k_cache || !v_cache || !tok_chunk || !tok_pos || !tok_score) return DELTAS_ERR_INVALID_ARGUMENT;
    if (n_new > 0 && (!k_new || !v_new || !aligned16(k_new) || !aligned16(v_new))) return DELTAS_ERR_INVALID_ARGUMENT;
    if (!aligned16(k_cache) || !aligned16(v_cache)) return DELTAS_ERR_INVALID_ARGUMENT;
    KvPlanes kv = make_planes(desc, k_cache, v_cache, tok_chunk, tok_pos);
    kv.tok_score = tok_score;
    return from_cuda(launch_append_kv_heads(kv, signal, cache_len, k_new, v_new, n_new, chunk_id, first_pos,
                                            as_stream(stream)));
}

size_t deltas_select_retain_heads_workspace_size(int32_t num_planes, int32_t cache_len) {
    if (num_planes < 0 || cache_len < 0) return 0;
    return select_heads_workspace_bytes(num_planes, cache_len);
}

deltas_status deltas_select_retain_heads(const deltas_policy* policy, int32_t num_planes, int32_t cache_len,
                                         int32_t plane_stride, const int32_t* tok_chunk, const float* tok_score,
                                         int32_t* retain_idx, int32_t* n_retained, uint8_t* mask,
                                         void* workspace, size_t workspace_bytes, void* stream)
{
    if (policy == nullptr || num_planes < 1 || cache_len < 0 || plane_stride < cache_len)
        return DELTAS_ERR_INVALID_ARGUMENT;
    const deltas_policy& p = *policy;
    if (p.budget_M < 1 || p.n_sink < 0 || p.n_window < 0 || p.n_buckets < 0) return DELTAS_ERR_INVALID_ARGUMENT;
    if ((long long)p.budget_M < (long long)p.n_sink + p.n_window + 1) return DELTAS_ERR_INVALID_ARGUMENT;
    if (p.n_buckets > 32) return DELTAS_ERR_UNSUPPORTED;
    if (cache_len > DELTAS_SELECT_MAX_CACHE_LEN || num_planes > 65535) return DELTAS_ERR_UNSUPPORTED;
    if (!retain_idx || !n_retained) return DELTAS_ERR_INVALID_ARGUMENT;
    if (cache_len > 0 && (!tok_chunk || !tok_score)) return DELTAS_ERR_INVALID_ARGUMENT;
    deltas_status st = check_workspace(workspace, workspace_bytes,
                                       deltas_select_retain_heads_workspace_size(num_planes, cache_len));
    if (st != DELTAS_OK) return st;
    return from_cuda(launch_select_heads(p, num_planes, cache_len, plane_stride, tok_chunk, tok_score, retain_idx,
                                         n_retained, mask, workspace, static_cast<int32_t*>(workspace),
                                         as_stream(stream)));
}

size_t deltas_compact_kv_heads_workspace_size(const deltas_kv_desc* desc, int32_t cache_len) {
    if (check_kv_desc(desc) != DELTAS_OK || cache_len < 0) return 0;
    KvPlanes kv = make_planes(desc, nullptr, nullptr, nullptr, nullptr);
    return compact_heads_workspace_bytes(kv, cache_len);
}

deltas_status deltas_compact_kv_heads(const deltas_kv_desc* desc, void* k_cache, void* v_cache,
                                      int32_t* tok_chunk, int32_t* tok_pos, float* tok_score,
                                      const int32_t* retain_idx, int32_t list_stride,
                                      const int32_t* n_retained, int32_t cache_len,
                                      void* workspace, size_t workspace_bytes, void* stream)
{
    deltas_status st = check_kv_desc(desc);
    if (st != DELTAS_OK) return st;
    if (cache_len < 0 || cache_len > desc->capacity || list_stride < 0) return DELTAS_ERR_INVALID_ARGUMENT;
    if (!k_cache || !v_cache || !tok_chunk || !tok_pos || !tok_score || !retain_idx || !n_retained)
        return DELTAS_ERR_INVALID_ARGUMENT;
    if (!aligned16(k_cache) || !aligned16(v_cache)) return DELTAS_ERR_INVALID_ARGUMENT;
    if (desc->num_layers * desc->num_kv_heads > 1 && list_stride < 1) return DELTAS_ERR_INVALID_ARGUMENT;
    st = check_workspace(workspace, workspace_bytes, deltas_compact_kv_heads_workspace_size(desc, cache_len));
    if (st != DELTAS_OK) return st;
    KvPlanes kv = make_planes(desc, k_cache, v_cache, tok_chunk, tok_pos);
    kv.tok_score = tok_score;
    return from_cuda(launch_compact_kv_heads(kv, retain_idx, list_stride, n_retained, cache_len, workspace,
                                             static_cast<int32_t*>(workspace), as_stream(stream)));
}

namespace {

// One batch of copies for a stream state.  per_head: the metadata rows (and the token scores) are
// [Lf][Hkv][capacity], one row of cache_len entries per plane, instead of one [capacity] row.
deltas_status copy_stream_state(const deltas_gdn_desc* gdn, const deltas_kv_desc* kv, int32_t cache_len,
                                int32_t n_chunks, const deltas_stream_buffers* src, const deltas_stream_buffers* dst,
                                const float* src_tok_score, float* dst_tok_score, bool per_head, void* stream)
{
    deltas_status st = check_gdn_desc(gdn);
    if (st != DELTAS_OK) return st;
    if (src == nullptr || dst == nullptr || n_chunks < 0) return DELTAS_ERR_INVALID_ARGUMENT;
    if (!src->state || !dst->state) return DELTAS_ERR_INVALID_ARGUMENT;
    if (n_chunks > 0 && (!src->chunk_scores || !dst->chunk_scores)) return DELTAS_ERR_INVALID_ARGUMENT;
    const void* cache_ptrs[8] = {src->k_cache, src->v_cache, src->tok_chunk, src->tok_pos,
                                 dst->k_cache, dst->v_cache, dst->tok_chunk, dst->tok_pos};
    if (kv == nullptr) {
        for (const void* p : cache_ptrs)
            if (p != nullptr) return DELTAS_ERR_INVALID_ARGUMENT;
    } else {
        st = check_kv_desc(kv);
        if (st != DELTAS_OK) return st;
        if (cache_len < 0 || cache_len > kv->capacity) return DELTAS_ERR_INVALID_ARGUMENT;
        for (const void* p : cache_ptrs)
            if (p == nullptr || !aligned16(p)) return DELTAS_ERR_INVALID_ARGUMENT;
        if (per_head) {             // per-plane metadata rows must start on 16-byte boundaries
            if (!src_tok_score || !dst_tok_score || !aligned16(src_tok_score) || !aligned16(dst_tok_score))
                return DELTAS_ERR_INVALID_ARGUMENT;
            if (kv->capacity % 4 != 0) return DELTAS_ERR_INVALID_ARGUMENT;
        }
    }
    if (per_head && kv == nullptr) return DELTAS_ERR_INVALID_ARGUMENT;
    if (!aligned16(src->state) || !aligned16(dst->state)) return DELTAS_ERR_INVALID_ARGUMENT;
    if (n_chunks > 0 && (!aligned16(src->chunk_scores) || !aligned16(dst->chunk_scores)))
        return DELTAS_ERR_INVALID_ARGUMENT;

    CopyBatch b;
    b.n = 0;
    auto add = [&](const void* from, void* to, uint64_t row_bytes, uint64_t stride, int64_t rows) {
        if (row_bytes == 0 || rows == 0) return;
        CopySeg& g = b.seg[b.n++];
        g.src = static_cast<const uint8_t*>(from); g.dst = static_cast<uint8_t*>(to);
        g.row_bytes = row_bytes; g.stride = stride; g.rows = rows;
    };
    add(src->state, dst->state,
        (uint64_t)gdn->num_layers * gdn->num_v_heads * gdn->value_dim * gdn->key_dim * 4, 0, 1);
    add(src->chunk_scores, dst->chunk_scores, (uint64_t)n_chunks * 4, 0, 1);
    if (kv != nullptr) {
        const uint64_t rb = (uint64_t)kv->head_dim * elt_bytes(kv->dtype);
        const int64_t planes = (int64_t)kv->num_layers * kv->num_kv_heads;
        add(src->k_cache, dst->k_cache, rb * cache_len, rb * kv->capacity, planes);
        add(src->v_cache, dst->v_cache, rb * cache_len, rb * kv->capacity, planes);
        const int64_t meta_rows = per_head ? planes : 1;
        const uint64_t meta_stride = per_head ? (uint64_t)kv->capacity * 4 : 0;
        add(src->tok_chunk, dst->tok_chunk, (uint64_t)cache_len * 4, meta_stride, meta_rows);
        add(src->tok_pos, dst->tok_pos, (uint64_t)cache_len * 4, meta_stride, meta_rows);
        if (per_head) add(src_tok_score, dst_tok_score, (uint64_t)cache_len * 4, meta_stride, meta_rows);
    }
    // no destination range may overlap a source range or another destination range
    auto extent_end = [](const CopySeg& g) { return (uint64_t)(g.rows - 1) * g.stride + g.row_bytes; };
    auto overlap = [](uintptr_t a0, uint64_t an, uintptr_t b0, uint64_t bn) {
        return a0 < b0 + bn && b0 < a0 + an;
    };
    for (int i = 0; i < b.n; ++i) {
        const uintptr_t d0 = reinterpret_cast<uintptr_t>(b.seg[i].dst);
        const uint64_t dn = extent_end(b.seg[i]);
        for (int j = 0; j < b.n; ++j) {
            if (overlap(d0, dn, reinterpret_cast<uintptr_t>(b.seg[j].src), extent_end(b.seg[j])))
                return DELTAS_ERR_INVALID_ARGUMENT;
            if (j != i && overlap(d0, dn, reinterpret_cast<uintptr_t>(b.seg[j].dst), extent_end(b.seg[j])))
                return DELTAS_ERR_INVALID_ARGUMENT;
        }
    }
    return from_cuda(launch_copy_batch(b, as_stream(stream)));
}

}  // namespace

deltas_status deltas_copy_stream_state(const deltas_gdn_desc* gdn, const deltas_kv_desc* kv,
                                       int32_t cache_len, int32_t n_chunks,
                                       const deltas_stream_buffers* src,
                                       const deltas_stream_buffers* dst, void* stream)
{
    return copy_stream_state(gdn, kv, cache_len, n_chunks, src, dst, nullptr, nullptr, false, stream);
}

deltas_status deltas_copy_stream_state_heads(const deltas_gdn_desc* gdn, const deltas_kv_desc* kv,
                                             int32_t cache_len, int32_t n_chunks,
                                             const deltas_stream_buffers* src,
                                             const deltas_stream_buffers* dst,
                                             const float* src_tok_score, float* dst_tok_score, void* stream)
{
    return copy_stream_state(gdn, kv, cache_len, n_chunks, src, dst, src_tok_score, dst_tok_score, true, stream);
}

deltas_status deltas_clear_device_status(void* workspace, void* stream) {
    if (workspace == nullptr) return DELTAS_ERR_WORKSPACE;
    return from_cuda(cudaMemsetAsync(workspace, 0, kStatusBytes, as_stream(stream)));
}

deltas_status deltas_set_wait_budget(void* workspace, uint32_t budget_ns, void* stream) {
    if (workspace == nullptr) return DELTAS_ERR_WORKSPACE;
    const uint32_t v = budget_ns;      // pageable source: copied before cudaMemcpyAsync returns
    return from_cuda(cudaMemcpyAsync(static_cast<uint8_t*>(workspace) + 8, &v, sizeof(v), cudaMemcpyHostToDevice,
                                     as_stream(stream)));
}

deltas_status deltas_get_device_status(const void* workspace, void* stream,
                                       int32_t* status_out, int32_t* detail_out)
{
    if (workspace == nullptr) return DELTAS_ERR_WORKSPACE;
    int32_t host[2] = {0, 0};
    cudaError_t e = cudaStreamSynchronize(as_stream(stream));
    if (e == cudaSuccess) e = cudaMemcpy(host, workspace, sizeof(host), cudaMemcpyDeviceToHost);
    if (e != cudaSuccess) return DELTAS_ERR_CUDA;
    if (status_out) *status_out = host[0];
    if (detail_out) *detail_out = host[1];
    return DELTAS_OK;
}

}  // extern "C"
