/*
 * deltas.h — C ABI of the DeltaS hot path on one GB300 GPU (sm_103a).
 *
 * DeltaS ("Reading the Gated Linear Attention State for KV Cache Eviction in Streaming Video")
 * scores each video chunk by the normalised change it causes in the gated-delta-rule recurrent
 * state (state drift, Sec. 3.2) and keeps the KV entries of high-drift chunks under a token
 * budget (Sec. 3.3, Alg. 1).  This library runs that path as CUDA kernels:
 *
 *   deltas_gdn_chunk_update  gated delta rule over a chunk (Eq. 1/2) + fused drift partials
 *   deltas_state_drift       drift partials from two stored states (Eq. 3 numerator/denominator)
 *   deltas_score_chunks      Delta S of Eq. 3 from the partials, stored as the chunk's score
 *   deltas_select_retain     sink / window / temporal spans / quota + fill (Sec. 3.3, Alg. 1)
 *   deltas_compact_kv        in-place, stream-order gather of the KV caches (Alg. 1, Sec. 3.3)
 *   deltas_append_kv         append a chunk's keys/values to the caches (Alg. 1 Prefill)
 *   deltas_*_heads           the same append / select / compact with a cache-internal token
 *                            signal (key norm, value norm; Sec. 4.3) ranked per KV head
 *
 * Conventions shared by every call
 * --------------------------------
 * - Tensor pointers are CUDA device memory owned by the caller, dense, in the layouts stated per
 *   call, 16-byte aligned.  The library allocates nothing and keeps no state between calls.
 * - `stream` is a cudaStream_t passed as void* (NULL = the legacy default stream).  Every call
 *   only enqueues work on it and returns at once; no call synchronises, except
 *   deltas_get_device_status.
 * - Scratch memory is a caller-provided `workspace` of at least the size reported by the matching
 *   deltas_*_workspace_size function, 256-byte aligned.  Its first 16 bytes are a sticky device
 *   status word: kernels that detect an error on the device (a bounded wait that ran out, an
 *   out-of-range index) record the first such error there and skip the unsafe part of their
 *   work.  Zero it once with deltas_clear_device_status before first use; read it with
 *   deltas_get_device_status.  Calls sharing a workspace must be ordered on one stream.  After a
 *   call that recorded an error, its outputs (and, for in-place calls, its in/out buffers) are
 *   unspecified: parts of the work may have completed before the error stopped the rest.
 * - Return value: DELTAS_OK when the work was enqueued; DELTAS_ERR_INVALID_ARGUMENT /
 *   DELTAS_ERR_UNSUPPORTED / DELTAS_ERR_WORKSPACE when the host-side checks reject the call
 *   (nothing is enqueued then); DELTAS_ERR_CUDA when a launch failed.  No exception crosses the
 *   ABI.
 */
#ifndef DELTAS_H
#define DELTAS_H

#include <stddef.h>
#include <stdint.h>

#if defined(__GNUC__)
#define DELTAS_API __attribute__((visibility("default")))
#else
#define DELTAS_API
#endif

#ifdef __cplusplus
extern "C" {
#endif

typedef enum deltas_status_e {
    DELTAS_OK = 0,
    DELTAS_ERR_INVALID_ARGUMENT = 1, /* a pointer, size or value outside its stated range        */
    DELTAS_ERR_UNSUPPORTED = 2,      /* valid, but a shape/dtype the library has no kernel for    */
    DELTAS_ERR_WORKSPACE = 3,        /* workspace missing, misaligned or smaller than required    */
    DELTAS_ERR_CUDA = 4,             /* a CUDA launch or runtime call failed                      */
    DELTAS_ERR_TIMEOUT = 5,          /* device: a bounded wait ran out (work skipped)             */
    DELTAS_ERR_DEVICE_INDEX = 6      /* device: an index array was out of range or out of order   */
} deltas_status;

typedef enum deltas_dtype_e {
    DELTAS_F32 = 0,  /* IEEE binary32 */
    DELTAS_BF16 = 1  /* bfloat16 */
} deltas_dtype;

/* Shape of the gated-delta (linear-attention) layers.  Value head h reads key head
 * floor(h * num_k_heads / num_v_heads) (grouped keys). */
typedef struct deltas_gdn_desc {
    int32_t num_layers;   /* L >= 1 */
    int32_t num_k_heads;  /* Hk >= 1 */
    int32_t num_v_heads;  /* Hv >= 1, a multiple of Hk */
    int32_t key_dim;      /* d_k in {16, 32, 64, 128} */
    int32_t value_dim;    /* d_v, equal to d_k (the only supported case) */
    int32_t dtype;        /* deltas_dtype of q, k, v and out; g, beta and the state are float32 */
    float q_scale;        /* read-out scale: o_t = q_scale * S_t q_t (commonly 1/sqrt(d_k)) */
} deltas_gdn_desc;

/* Retention policy (Alg. 1 inputs; Sec. 3.3). */
typedef struct deltas_policy {
    int32_t budget_M;   /* M >= n_sink + n_window + 1: tokens kept per full-attention layer */
    int32_t n_sink;     /* n_s >= 0: first slots always kept (attention sinks) */
    int32_t n_window;   /* n_w >= 0: most recent slots always kept */
    int32_t n_buckets;  /* N in [0, 32]: equal temporal spans; 0 means no bucketing (= 1 span) */
} deltas_policy;

/* Shape of the full-attention KV caches: K and V are separate buffers, each
 * [num_layers][num_kv_heads][capacity][head_dim] of dtype; a (layer, head) pair is one "plane"
 * of `capacity` rows of head_dim elements. */
typedef struct deltas_kv_desc {
    int32_t num_layers;    /* Lf >= 1 */
    int32_t num_kv_heads;  /* Hkv >= 1 */
    int32_t head_dim;      /* D >= 1; head_dim * element size must be a multiple of 16 bytes */
    int32_t dtype;         /* deltas_dtype of the caches */
    int32_t capacity;      /* rows allocated per plane (>= the largest cache_len used) */
} deltas_kv_desc;

/* ------------------------------------------------------------------------------------------ */
/* Version and status text                                                                     */
/* ------------------------------------------------------------------------------------------ */

/* Static string "deltas <major>.<minor>.<patch> sm_103a". */
DELTAS_API const char* deltas_version(void);

/* Static, never NULL, description of a deltas_status value (unknown codes included). */
DELTAS_API const char* deltas_status_string(int32_t status);

/* ------------------------------------------------------------------------------------------ */
/* Gated delta rule over one chunk, with the state drift partials fused in.                    */
/*                                                                                              */
/* Paper: Sec. 3.2, Eq. 1 S_t = S_{t-1}(alpha_t (I - beta_t k_t k_t^T)) + beta_t v_t k_t^T     */
/* (equivalently Eq. 2), run over the n_tokens tokens of one video chunk in stream order for   */
/* every layer and value head; the state before the chunk is S_before and the state after it   */
/* S_after of Eq. 3.  Alg. 1: "Prefill(c) updates S"; the read-out o_t = q_scale S_t q_t is     */
/* the layer output of that prefill.                                                            */
/*                                                                                              */
/*   q, k   [L][n_tokens][Hk][d_k]  dtype   keys L2-normalised by the caller; q may be NULL     */
/*                                          when out is NULL                                   */
/*   v      [L][n_tokens][Hv][d_v]  dtype                                                      */
/*   g      [L][n_tokens][Hv]       float   log decay, alpha_t = exp(g_t), g_t <= 0 expected    */
/*   beta   [L][n_tokens][Hv]       float   write strength in [0, 1]                           */
/*   state  [L][Hv][d_v][d_k]       float   in: S_before, out: S_after (updated in place)      */
/*   out    [L][n_tokens][Hv][d_v]  dtype   o_t after each token's update; NULL to skip        */
/*   drift_partials [L][Hv][2]      float   NULL to skip; else [l][h][0] = sum (S_after -      */
/*                                          S_before)^2 and [l][h][1] = sum S_before^2 over    */
/*                                          the head's d_v x d_k entries                       */
/* n_tokens = 0 leaves the state unchanged (partials then hold 0 and ||S_before||^2).          */
/* Errors: INVALID_ARGUMENT for NULL/misaligned pointers, negative sizes or Hv % Hk != 0;      */
/* UNSUPPORTED for d_k != d_v or d_k outside {16,32,64,128}; WORKSPACE for a short workspace. */
/* Workspace: the status word plus, for d = 128 bf16, the per-tile factors of the chunkwise     */
/* form (16,656 bytes per layer, value head and 64-token tile; 16,912 with the read-out),       */
/* written and read within the call.  A call with out != NULL needs                            */
/* deltas_gdn_chunk_update_readout_workspace_size bytes: for d = 128 bf16 that adds each       */
/* token's write u_t (512 bytes per token and value head) and the state at the start of every  */
/* 128-token block (64 KiB per block and value head); a shorter workspace returns WORKSPACE.   */
/* Kernels: d = 128 bfloat16 runs on the tensor cores (a factor kernel, a state-chain kernel   */
/* and, with out != NULL, a read-out kernel that forms each 128-token block's outputs from the */
/* block's starting state and writes; when few heads leave most SMs idle and neither out nor  */
/* write sizes are asked for, the chain runs each head's tiles as two segments on three CTAs, */
/* the first joining them at its end), or returns UNSUPPORTED when that path cannot be launched */
/* (no silent fallback).  Every other shape runs token by token on the CUDA cores.            */
/* ------------------------------------------------------------------------------------------ */
DELTAS_API size_t deltas_gdn_chunk_update_workspace_size(const deltas_gdn_desc* desc, int32_t n_tokens);

/* Workspace bytes for a deltas_gdn_chunk_update(_write_norms) call that passes out != NULL    */
/* (>= deltas_gdn_chunk_update_workspace_size; equal to it except for d = 128 bfloat16).      */
DELTAS_API size_t deltas_gdn_chunk_update_readout_workspace_size(const deltas_gdn_desc* desc, int32_t n_tokens);

DELTAS_API deltas_status deltas_gdn_chunk_update(const deltas_gdn_desc* desc, int32_t n_tokens,
                                      const void* q, const void* k, const void* v,
                                      const float* g, const float* beta,
                                      float* state, void* out, float* drift_partials,
                                      void* workspace, size_t workspace_bytes, void* stream);

/* ------------------------------------------------------------------------------------------ */
/* The same update, also returning the comparison signal of Sec. 4.3 (the write size of HOLA's */
/* score, as the appendix describes it): the rank-one write of token t is u_t k_t^T with        */
/* u_t = beta_t (v_t - alpha_t S_{t-1} k_t), of Frobenius norm ||u_t||_2 for a unit key.        */
/*   write_norms [L][Hv] float  (required here) receives per (layer, value head) the sum over  */
/*                              the n_tokens tokens of beta_t ||v_t - alpha_t S_{t-1} k_t||_2    */
/* (0 for n_tokens = 0).  Every other argument, result and error as deltas_gdn_chunk_update;    */
/* INVALID_ARGUMENT also for a NULL or misaligned write_norms.  On the tensor-core path a tile  */
/* whose decay over its 64 tokens exp(G_C) is below 2^-60 (G_C < -41.6) adds nothing.          */
/* ------------------------------------------------------------------------------------------ */
DELTAS_API deltas_status deltas_gdn_chunk_update_write_norms(const deltas_gdn_desc* desc, int32_t n_tokens,
                                      const void* q, const void* k, const void* v,
                                      const float* g, const float* beta,
                                      float* state, void* out, float* drift_partials,
                                      float* write_norms, void* workspace,
                                      size_t workspace_bytes, void* stream);

/* The comparison signal's chunk score: write sizes averaged over heads, layers and the chunk's */
/* n_tokens tokens, chunk_scores[chunk_id] = sum(write_norms) / (L * Hv * n_tokens), 0 when     */
/* n_tokens = 0 (float32; the sum is taken in double on the device).                           */
/* Errors: INVALID_ARGUMENT for NULL pointers or negative sizes / chunk_id.                     */
DELTAS_API deltas_status deltas_score_write_norms(int32_t num_layers, int32_t num_v_heads,
                                      const float* write_norms, int32_t n_tokens,
                                      int32_t chunk_id, float* chunk_scores, void* stream);

/* ------------------------------------------------------------------------------------------ */
/* State drift partials from two stored states (Sec. 3.2, Eq. 3 numerator and denominator per  */
/* layer and head; the paper keeps a copy of the previous state for this, Sec. 3.2).           */
/*   s_before, s_after [L][Hv][d_v][d_k] float;  drift_partials [L][Hv][2] float (as above).   */
/* Only num_layers, num_v_heads, key_dim and value_dim of desc are used.                       */
/* ------------------------------------------------------------------------------------------ */
DELTAS_API size_t deltas_state_drift_workspace_size(const deltas_gdn_desc* desc);

DELTAS_API deltas_status deltas_state_drift(const deltas_gdn_desc* desc, const float* s_before,
                                 const float* s_after, float* drift_partials,
                                 void* workspace, size_t workspace_bytes, void* stream);

/* ------------------------------------------------------------------------------------------ */
/* Chunk score (Sec. 3.2, Eq. 3; Alg. 1 "Delta S <- mean_i ||S^i - S^i_before|| /             */
/* ||S^i_before||" and "score[t] <- Delta S"):                                                  */
/*   Delta S = (1/L) sum_l sqrt(sum_h partials[l][h][0]) / sqrt(sum_h partials[l][h][1])       */
/* The per-layer norm runs over all heads of the layer.  A layer whose denominator is 0        */
/* contributes 0 when its numerator is 0 and +infinity otherwise.  The reduction order is       */
/* fixed (deterministic): per-layer sums over the heads in float (pairwise tree), each layer's   */
/* square roots and quotient in float (correctly rounded), the mean over layers in double; the  */
/* score is stored as float to chunk_scores[chunk_id] (device memory, [>= chunk_id + 1]).       */
/* ------------------------------------------------------------------------------------------ */
DELTAS_API deltas_status deltas_score_chunks(int32_t num_layers, int32_t num_v_heads,
                                  const float* drift_partials, int32_t chunk_id,
                                  float* chunk_scores, void* stream);

/* ------------------------------------------------------------------------------------------ */
/* Retain selection (Sec. 3.3; Alg. 1 eviction branch).                                        */
/*                                                                                              */
/* The cache holds cache_len slots in stream order; tok_chunk[i] is the arrival chunk of slot  */
/* i and chunk_scores[c] the stored score of chunk c (shared by all its tokens).  If cache_len  */
/* <= M every slot is kept.  Otherwise the first n_s and the last n_w slots are kept; the rest  */
/* (candidates) are split into N equal spans of arrival chunk,                                  */
/*   span(i) = floor((tok_chunk[i] - c_lo) * N / (c_hi - c_lo + 1)),                            */
/* c_lo/c_hi the smallest/largest candidate chunk; each span keeps its best                     */
/* min(floor((M - n_s - n_w) / N), |span|) candidates and the remaining capacity goes to the    */
/* best remaining candidates.  "Best" = higher score under the IEEE-754 total order of float,  */
/* ties to the earlier slot.                                                                    */
/*                                                                                              */
/*   tok_chunk   [cache_len] int32 in [0, num_chunks)      chunk_scores [num_chunks] float     */
/*   retain_idx  [min(cache_len, M)] int32  out: kept slots, strictly ascending                 */
/*   n_retained  [1] int32 (device)         out: min(cache_len, M)                              */
/*   mask        [cache_len] uint8          out: 1 = kept, 0 = evicted; NULL to skip            */
/* A tok_chunk value outside [0, num_chunks) is reported as DEVICE_INDEX in the status word    */
/* (outputs are then unspecified).  cache_len above DELTAS_SELECT_MAX_CACHE_LEN (2^20) returns   */
/* UNSUPPORTED.                                                                                 */
/* ------------------------------------------------------------------------------------------ */
#define DELTAS_SELECT_MAX_CACHE_LEN 1048576

DELTAS_API size_t deltas_select_retain_workspace_size(int32_t cache_len);

DELTAS_API deltas_status deltas_select_retain(const deltas_policy* policy, int32_t cache_len,
                                   int32_t num_chunks, const int32_t* tok_chunk,
                                   const float* chunk_scores, int32_t* retain_idx,
                                   int32_t* n_retained, uint8_t* mask,
                                   void* workspace, size_t workspace_bytes, void* stream);

/* ------------------------------------------------------------------------------------------ */
/* Retain selection without a caller workspace (the paper has no counterpart: this is a         */
/* library convenience).  For callers that may not allocate device memory: a serving runtime    */
/* that owns all of HBM through its own pool, or code running where cudaMalloc is not allowed.  */
/* It calls no cudaMalloc, cudaFree or other allocating routine.                                */
/*                                                                                              */
/* Arguments, outputs and results are those of deltas_select_retain without the workspace.  The */
/* scratch is a fixed device array inside the library sized for                                 */
/* DELTAS_SELECT_STATIC_MAX_CACHE_LEN slots (about 2.25 MiB); a larger cache_len returns        */
/* DELTAS_ERR_UNSUPPORTED with nothing enqueued.                                                */
/*   - Every call looks up the array's address in the current context (the stream must belong  */
/*     to the current device); the first call on a device loads the library's module there, so */
/*     make it before any stream capture.                                                       */
/*   - All calls on a device share the array.  Calls whose kernels may run at the same time on   */
/*     the GPU (streams with no ordering between them) race and give undefined results.         */
/*   - Each call clears the status word at the head of the array on its stream before the       */
/*     launch.  A tok_chunk value outside [0, num_chunks) is reported on the device by          */
/*     *n_retained == 0 while cache_len > 0 (a valid call always keeps at least one slot).      */
/* ------------------------------------------------------------------------------------------ */
#define DELTAS_SELECT_STATIC_MAX_CACHE_LEN 65536

DELTAS_API deltas_status deltas_select_retain_static(const deltas_policy* policy, int32_t cache_len,
                                   int32_t num_chunks, const int32_t* tok_chunk,
                                   const float* chunk_scores, int32_t* retain_idx,
                                   int32_t* n_retained, uint8_t* mask, void* stream);

/* ------------------------------------------------------------------------------------------ */
/* In-place KV compaction (Alg. 1 "KV <- KV[I_sink u I_DeltaS u I_window]", applied to every    */
/* full-attention layer; Sec. 3.3: survivors keep their original position indices).            */
/*                                                                                              */
/* For every plane of k_cache and v_cache, and for tok_chunk and tok_pos ([capacity] int32):    */
/*   row[j] <- row[retain_idx[j]]   for j < *n_retained,  in place;                             */
/* rows at and past *n_retained are not written.  retain_idx is read on the device and must be  */
/* strictly ascending with j <= retain_idx[j] < cache_len (as deltas_select_retain writes it);  */
/* otherwise nothing is moved and DEVICE_INDEX is recorded.  Positions in tok_pos are moved,    */
/* never renumbered.  cache_len <= capacity.                                                    */
/* ------------------------------------------------------------------------------------------ */
DELTAS_API size_t deltas_compact_kv_workspace_size(const deltas_kv_desc* desc, int32_t cache_len);

DELTAS_API deltas_status deltas_compact_kv(const deltas_kv_desc* desc, void* k_cache, void* v_cache,
                                int32_t* tok_chunk, int32_t* tok_pos,
                                const int32_t* retain_idx, const int32_t* n_retained,
                                int32_t cache_len, void* workspace, size_t workspace_bytes,
                                void* stream);

/* ------------------------------------------------------------------------------------------ */
/* Append one chunk to the caches (Alg. 1 "Prefill(c) ... appends c to KV").                   */
/*   k_new, v_new [Lf][Hkv][n_new][D] dtype: the chunk's keys/values of every layer;            */
/*   rows cache_len .. cache_len + n_new - 1 of every plane receive them, tok_chunk of those    */
/*   slots is set to chunk_id and tok_pos to first_pos, first_pos + 1, ...                      */
/* Errors: INVALID_ARGUMENT if cache_len + n_new > capacity or a size is negative.             */
/* ------------------------------------------------------------------------------------------ */
DELTAS_API deltas_status deltas_append_kv(const deltas_kv_desc* desc, void* k_cache, void* v_cache,
                               int32_t* tok_chunk, int32_t* tok_pos, int32_t cache_len,
                               const void* k_new, const void* v_new, int32_t n_new,
                               int32_t chunk_id, int32_t first_pos, void* stream);

/* ------------------------------------------------------------------------------------------ */
/* Question-time snapshot and restore (Sec. 3.3, "Question answering": before a question the  */
/* stream state, both memories, is saved; after the answer it is restored together with the    */
/* retention scores and chunk indices, so that question turns leave the stream unchanged).      */
/*                                                                                              */
/* A stream state is the set of buffers below.  src and dst are two such sets laid out by the  */
/* same descriptors (snapshot: live -> saved copy; restore: saved copy -> live):                */
/*   state          [L][Hv][d_v][d_k] fp32 (gdn desc)             copied whole;                  */
/*   chunk_scores   fp32                                          entries 0 .. n_chunks - 1;     */
/*   k_cache, v_cache [Lf][Hkv][capacity][D] (kv desc dtype)      rows 0 .. cache_len - 1 of     */
/*                                                                every plane;                   */
/*   tok_chunk, tok_pos [capacity] int32                          entries 0 .. cache_len - 1.    */
/* kv == NULL copies state and scores only; the four cache pointers of both sets must then be  */
/* NULL.  That is enough when the question appends to the caches but evicts nothing: the rows  */
/* it appends lie past cache_len, which the caller restores on the host along with the stream  */
/* position and the chunk counter (the library keeps none of them).  Everything moves in one    */
/* kernel launch on `stream`, 16 bytes per load and store; the sets must not overlap.           */
/* Errors (nothing enqueued): INVALID_ARGUMENT for a NULL required pointer, a pointer that is   */
/* not 16-byte aligned, n_chunks < 0, cache_len outside [0, capacity], or overlapping source   */
/* and destination ranges; the descriptor checks of the other calls.                           */
/* ------------------------------------------------------------------------------------------ */
typedef struct {
    float* state;
    float* chunk_scores;
    void* k_cache;
    void* v_cache;
    int32_t* tok_chunk;
    int32_t* tok_pos;
} deltas_stream_buffers;

DELTAS_API deltas_status deltas_copy_stream_state(const deltas_gdn_desc* gdn, const deltas_kv_desc* kv,
                                       int32_t cache_len, int32_t n_chunks,
                                       const deltas_stream_buffers* src,
                                       const deltas_stream_buffers* dst, void* stream);

/* The same for a stream ranked by a per-head token signal (deltas_*_heads): tok_chunk and tok_pos */
/* of both sets are [Lf][Hkv][capacity] and every plane's entries 0 .. cache_len - 1 are copied,   */
/* as are those of the token scores src_tok_score -> dst_tok_score ([Lf][Hkv][capacity] float).   */
/* kv is required, and kv->capacity must be a multiple of 4 (each plane's metadata row then starts */
/* on a 16-byte boundary); otherwise, and for the reasons above, INVALID_ARGUMENT.                 */
DELTAS_API deltas_status deltas_copy_stream_state_heads(const deltas_gdn_desc* gdn, const deltas_kv_desc* kv,
                                             int32_t cache_len, int32_t n_chunks,
                                             const deltas_stream_buffers* src,
                                             const deltas_stream_buffers* dst,
                                             const float* src_tok_score, float* dst_tok_score,
                                             void* stream);

/* ------------------------------------------------------------------------------------------ */
/* Per-head token signals (Sec. 4.3, the controlled comparison of retention signals, and the   */
/* appendix table of signals).  Instead of one score per chunk, every cached token of every     */
/* (layer, KV head) plane carries its own score, read from the cache rows themselves:           */
/*   DELTAS_SIGNAL_KEY_NORM    score = -||k||_2 of the token's key row   (key-norm signal)      */
/*   DELTAS_SIGNAL_VALUE_NORM  score = +||v||_2 of the token's value row (value-norm signal)    */
/* Each plane is ranked on its own under the policy of deltas_select_retain, so every plane     */
/* keeps its own min(cache_len, M) tokens; the per-slot metadata is therefore per plane:        */
/*   tok_chunk, tok_pos [Lf][Hkv][capacity] int32    tok_score [Lf][Hkv][capacity] float       */
/* (plane p = layer * Hkv + head).  All planes hold the same number of tokens, cache_len.       */
/* ------------------------------------------------------------------------------------------ */
typedef enum deltas_signal_e {
    DELTAS_SIGNAL_KEY_NORM = 1,
    DELTAS_SIGNAL_VALUE_NORM = 2
} deltas_signal;

/* Append one chunk and score its tokens: as deltas_append_kv, and in every plane p the new     */
/* slots get tok_chunk[p][.] = chunk_id, tok_pos[p][.] = first_pos, first_pos + 1, ... and      */
/* tok_score[p][.] = the signal of the row just stored (squares summed in float32 from the      */
/* stored values, then a correctly rounded square root).  A token's score depends on its row    */
/* alone, so it is computed once, here, and moved with the row by deltas_compact_kv_heads; it   */
/* equals the score recomputed from the cache at eviction time.                                 */
/* Errors: those of deltas_append_kv; INVALID_ARGUMENT for an unknown signal or a NULL          */
/* tok_score.                                                                                   */
DELTAS_API deltas_status deltas_append_kv_heads(const deltas_kv_desc* desc, int32_t signal,
                                     void* k_cache, void* v_cache, int32_t* tok_chunk,
                                     int32_t* tok_pos, float* tok_score, int32_t cache_len,
                                     const void* k_new, const void* v_new, int32_t n_new,
                                     int32_t chunk_id, int32_t first_pos, void* stream);

/* Per-plane retain selection: for each of the num_planes planes, the rule of                   */
/* deltas_select_retain with the slot's own score tok_score[p][i] in place of its chunk's      */
/* (spans still split the candidates' arrival chunks tok_chunk[p][.], computed per plane).      */
/*   tok_chunk, tok_score  [num_planes][plane_stride], slots 0 .. cache_len - 1 read             */
/*   retain_idx  [num_planes][M] int32  out: row p = the kept slots of plane p, ascending        */
/*   n_retained  [1] int32 (device)     out: min(cache_len, M), the same for every plane        */
/*   mask        [num_planes][plane_stride] uint8  out: 1 = kept; NULL to skip                   */
/* A cluster of four CTAs ranks one plane, each CTA a quarter of its candidates (a radix select */
/* on the score's total-order bits, then on the slot for ties, with the four CTAs' counts added */
/* through distributed shared memory); the keys sit in shared memory when they fit, else in the  */
/* workspace.  The launch needs four SMs of one GPC free at once for each cluster: a context    */
/* limited to fewer SMs than that gets the launch error back (DELTAS_ERR_CUDA).                 */
/* A negative tok_chunk value is reported as DEVICE_INDEX.  cache_len above                     */
/* DELTAS_SELECT_MAX_CACHE_LEN or plane_stride < cache_len: UNSUPPORTED / INVALID_ARGUMENT.     */
DELTAS_API size_t deltas_select_retain_heads_workspace_size(int32_t num_planes, int32_t cache_len);

DELTAS_API deltas_status deltas_select_retain_heads(const deltas_policy* policy, int32_t num_planes,
                                         int32_t cache_len, int32_t plane_stride,
                                         const int32_t* tok_chunk, const float* tok_score,
                                         int32_t* retain_idx, int32_t* n_retained, uint8_t* mask,
                                         void* workspace, size_t workspace_bytes, void* stream);

/* Per-plane in-place compaction: as deltas_compact_kv, except that plane p of k_cache and      */
/* v_cache and row p of tok_chunk, tok_pos and tok_score ([Lf][Hkv][capacity]) are gathered by */
/* their own list, row p of retain_idx ([Lf * Hkv][list_stride], list_stride >= *n_retained).   */
/* Every list must be strictly ascending with j <= retain_idx[p][j] < cache_len; otherwise      */
/* nothing is moved and DEVICE_INDEX is recorded.                                               */
DELTAS_API size_t deltas_compact_kv_heads_workspace_size(const deltas_kv_desc* desc, int32_t cache_len);

DELTAS_API deltas_status deltas_compact_kv_heads(const deltas_kv_desc* desc, void* k_cache, void* v_cache,
                                      int32_t* tok_chunk, int32_t* tok_pos, float* tok_score,
                                      const int32_t* retain_idx, int32_t list_stride,
                                      const int32_t* n_retained, int32_t cache_len,
                                      void* workspace, size_t workspace_bytes, void* stream);

/* ------------------------------------------------------------------------------------------ */
/* Device status word (first 16 bytes of a workspace).                                          */
/* ------------------------------------------------------------------------------------------ */

/* Enqueue a zeroing of the status word. */
DELTAS_API deltas_status deltas_clear_device_status(void* workspace, void* stream);

/* Enqueue on `stream` a write of the workspace's bounded-wait budget (word 2 of the status
 * header): a wait bounded by it gives up after `budget_ns` nanoseconds (0, the value
 * deltas_clear_device_status leaves: about one second) and records DELTAS_ERR_TIMEOUT; the other
 * roles of that kernel then stop at their next wait, drain the copies and MMAs they issued (those
 * drains keep the one-second bound) and return.  It bounds every wait of the selection and
 * compaction kernels, and the first wait of each kernel of deltas_gdn_chunk_update (the factor
 * kernel's first key tile, the state chain's first value tile, the read-out's first query and key
 * blocks); the per-tile waits of the update keep the one-second bound, since a bound read at run
 * time there made the latency-bound state chain about 5 % slower.  Not a paper operation: a wait
 * that runs out is the library's answer to a peer that never arrives (a CTA that cannot become
 * resident, say), and a small budget lets a test make that path run.  The host value is copied
 * before the call returns. */
DELTAS_API deltas_status deltas_set_wait_budget(void* workspace, uint32_t budget_ns, void* stream);

/* Synchronise `stream`, then read the status word: *status_out = first recorded deltas_status
 * (DELTAS_OK if none), *detail_out = kernel-specific detail (e.g. the offending index); either
 * output pointer may be NULL. */
DELTAS_API deltas_status deltas_get_device_status(const void* workspace, void* stream,
                                       int32_t* status_out, int32_t* detail_out);

#ifdef __cplusplus
}
#endif

#endif /* DELTAS_H */
