/*
 * DeltaS CPU oracle — plain, slow, obviously-correct fp64 reference of the hot path.
 *
 * TEST INFRASTRUCTURE ONLY.  Only the test-suite, the smoke check and the CPU-baseline leg of
 * the benchmark call this file.  It shares no code, header, table or helper with the CUDA
 * library, and nothing in the CUDA library calls it.
 *
 * Paper: "DeltaS: Reading the Gated Linear Attention State for KV Cache Eviction in Streaming
 * Video".  Every function cites the passage it follows.
 *
 * Conventions (all arrays dense, row-major, element counts not bytes):
 *   q, k  : [L][T][Hk][dk]   float   (bf16 inputs are widened to float by the caller, exactly)
 *   v     : [L][T][Hv][dv]   float
 *   g     : [L][T][Hv]       float   log of the decay alpha_t (alpha_t = exp(g_t))
 *   beta  : [L][T][Hv]       float   write strength beta_t
 *   S     : [L][Hv][dv][dk]  double  state, rows = value dimension, columns = key dimension
 *   out   : [L][T][Hv][dv]   double  o_t = q_scale * S_t q_t  (optional)
 *   Value head h reads key head floor(h * Hk / Hv) (grouped keys).
 *
 * All arithmetic is fp64; inputs are the exact values the GPU reads.
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

#define ORACLE_OK 0
#define ORACLE_BAD_ARG 1
#define ORACLE_NO_MEMORY 2

/* ------------------------------------------------------------------------------------------ */
/* Gated delta rule, residual form (Sec. 3.2, Eq. 2):                                          */
/*     S_t = alpha_t S_{t-1} + beta_t (v_t - alpha_t S_{t-1} k_t) k_t^T                         */
/* processed token by token in stream order.  If out != NULL, o_t = q_scale * S_t q_t is        */
/* written after the update of token t (the read-out of the prefill, Alg. 1 "Prefill").        */
/* If wnorm != NULL ([L][Hv]), it receives per (layer, head) the sum over the chunk's tokens of */
/* the write size beta_t ||v_t - alpha_t S_{t-1} k_t||_2 (the comparison signal of Sec. 4.3 and */
/* the appendix's description of it: the residual times the write strength, per head).         */
/* ------------------------------------------------------------------------------------------ */
int oracle_gdn_recurrence(int L, int Hk, int Hv, int dk, int dv, int T,
                          const float* q, const float* k, const float* v,
                          const float* g, const float* beta,
                          double* S, double* out, double q_scale, double* wnorm)
{
    if (L < 1 || Hk < 1 || Hv < 1 || dk < 1 || dv < 1 || T < 0 || Hv % Hk != 0) return ORACLE_BAD_ARG;
    if (!k || !v || !g || !beta || !S || (out && !q)) return ORACLE_BAD_ARG;
    double* r = (double*)malloc(sizeof(double) * (size_t)dv);
    if (!r) return ORACLE_NO_MEMORY;
    if (wnorm) memset(wnorm, 0, sizeof(double) * (size_t)L * Hv);
    for (int l = 0; l < L; ++l) {
        for (int h = 0; h < Hv; ++h) {
            const int kh = (int)(((long long)h * Hk) / Hv);
            double* Sh = S + ((size_t)l * Hv + h) * (size_t)dv * dk;
            for (int t = 0; t < T; ++t) {
                const size_t kofs = (((size_t)l * T + t) * Hk + kh) * (size_t)dk;
                const size_t vofs = (((size_t)l * T + t) * Hv + h) * (size_t)dv;
                const size_t gofs = ((size_t)l * T + t) * Hv + h;
                const float* kt = k + kofs;
                const float* vt = v + vofs;
                const double alpha = exp((double)g[gofs]);
                const double b = (double)beta[gofs];
                /* r = S_{t-1} k_t, read from the state before this token's write */
                for (int i = 0; i < dv; ++i) {
                    double acc = 0.0;
                    for (int j = 0; j < dk; ++j) acc += Sh[(size_t)i * dk + j] * (double)kt[j];
                    r[i] = acc;
                }
                /* S_t = alpha S_{t-1} + u k^T  with  u = beta (v - alpha r) */
                double uu = 0.0;
                for (int i = 0; i < dv; ++i) {
                    const double u = b * ((double)vt[i] - alpha * r[i]);
                    uu += u * u;
                    for (int j = 0; j < dk; ++j)
                        Sh[(size_t)i * dk + j] = alpha * Sh[(size_t)i * dk + j] + u * (double)kt[j];
                }
                if (wnorm) wnorm[(size_t)l * Hv + h] += sqrt(uu);
                if (out) {
                    const float* qt = q + kofs;
                    double* ot = out + vofs;
                    for (int i = 0; i < dv; ++i) {
                        double acc = 0.0;
                        for (int j = 0; j < dk; ++j) acc += Sh[(size_t)i * dk + j] * (double)qt[j];
                        ot[i] = q_scale * acc;
                    }
                }
            }
        }
    }
    free(r);
    return ORACLE_OK;
}

/* ------------------------------------------------------------------------------------------ */
/* Gated delta rule, product form (Sec. 3.2, Eq. 1):                                           */
/*     S_t = S_{t-1} (alpha_t (I - beta_t k_t k_t^T)) + beta_t v_t k_t^T                       */
/* written literally with a dk x dk transition matrix.  O(dk^3) per token: used only as a      */
/* self-check of the residual form on small inputs.  Same layouts as oracle_gdn_recurrence.    */
/* ------------------------------------------------------------------------------------------ */
int oracle_gdn_recurrence_product_form(int L, int Hk, int Hv, int dk, int dv, int T,
                                       const float* k, const float* v,
                                       const float* g, const float* beta, double* S)
{
    if (L < 1 || Hk < 1 || Hv < 1 || dk < 1 || dv < 1 || T < 0 || Hv % Hk != 0) return ORACLE_BAD_ARG;
    if (!k || !v || !g || !beta || !S) return ORACLE_BAD_ARG;
    double* P = (double*)malloc(sizeof(double) * (size_t)dk * dk);
    double* N = (double*)malloc(sizeof(double) * (size_t)dv * dk);
    if (!P || !N) { free(P); free(N); return ORACLE_NO_MEMORY; }
    for (int l = 0; l < L; ++l) {
        for (int h = 0; h < Hv; ++h) {
            const int kh = (int)(((long long)h * Hk) / Hv);
            double* Sh = S + ((size_t)l * Hv + h) * (size_t)dv * dk;
            for (int t = 0; t < T; ++t) {
                const float* kt = k + (((size_t)l * T + t) * Hk + kh) * (size_t)dk;
                const float* vt = v + (((size_t)l * T + t) * Hv + h) * (size_t)dv;
                const size_t gofs = ((size_t)l * T + t) * Hv + h;
                const double alpha = exp((double)g[gofs]);
                const double b = (double)beta[gofs];
                /* P = alpha (I - b k k^T) */
                for (int a = 0; a < dk; ++a)
                    for (int c = 0; c < dk; ++c)
                        P[(size_t)a * dk + c] = alpha * ((a == c ? 1.0 : 0.0) - b * (double)kt[a] * (double)kt[c]);
                /* N = S P + b v k^T */
                for (int i = 0; i < dv; ++i)
                    for (int c = 0; c < dk; ++c) {
                        double acc = 0.0;
                        for (int a = 0; a < dk; ++a) acc += Sh[(size_t)i * dk + a] * P[(size_t)a * dk + c];
                        N[(size_t)i * dk + c] = acc + b * (double)vt[i] * (double)kt[c];
                    }
                memcpy(Sh, N, sizeof(double) * (size_t)dv * dk);
            }
        }
    }
    free(P);
    free(N);
    return ORACLE_OK;
}

/* ------------------------------------------------------------------------------------------ */
/* State-drift partial sums (Sec. 3.2, Eq. 3 numerator and denominator, per layer and head):   */
/*     partials[l][h][0] = sum over the head's dv x dk entries of (S_after - S_before)^2        */
/*     partials[l][h][1] = sum of S_before^2                                                    */
/* The per-layer Frobenius norms of Eq. 3 run over all heads of the layer, so they are the      */
/* square roots of the per-layer sums of these partials.                                        */
/* ------------------------------------------------------------------------------------------ */
int oracle_drift_partials(int L, int Hv, int dv, int dk,
                          const double* s_before, const double* s_after, double* partials)
{
    if (L < 1 || Hv < 1 || dv < 1 || dk < 1 || !s_before || !s_after || !partials) return ORACLE_BAD_ARG;
    const size_t hs = (size_t)dv * dk;
    for (int l = 0; l < L; ++l)
        for (int h = 0; h < Hv; ++h) {
            const double* b = s_before + ((size_t)l * Hv + h) * hs;
            const double* a = s_after + ((size_t)l * Hv + h) * hs;
            double num = 0.0, den = 0.0;
            for (size_t e = 0; e < hs; ++e) {
                const double d = a[e] - b[e];
                num += d * d;
                den += b[e] * b[e];
            }
            partials[((size_t)l * Hv + h) * 2 + 0] = num;
            partials[((size_t)l * Hv + h) * 2 + 1] = den;
        }
    return ORACLE_OK;
}

/* ------------------------------------------------------------------------------------------ */
/* Chunk score (Sec. 3.2, Eq. 3; Alg. 1 "Delta S <- mean_i ..."):                               */
/*     Delta S = (1/L) sum_l ||S^l_after - S^l_before||_F / ||S^l_before||_F                    */
/* with the per-layer norms taken over all heads.  The paper leaves ||S_before|| = 0 open; the  */
/* reading used here: a layer with zero numerator and zero denominator contributes 0, a layer   */
/* with zero denominator and positive numerator contributes +infinity (a chunk written into an  */
/* empty state is maximally new).                                                               */
/* ------------------------------------------------------------------------------------------ */
double oracle_chunk_score(int L, int Hv, const double* partials)
{
    double total = 0.0;
    for (int l = 0; l < L; ++l) {
        double num = 0.0, den = 0.0;
        for (int h = 0; h < Hv; ++h) {
            num += partials[((size_t)l * Hv + h) * 2 + 0];
            den += partials[((size_t)l * Hv + h) * 2 + 1];
        }
        double term;
        if (den > 0.0) term = sqrt(num) / sqrt(den);
        else term = (num > 0.0) ? INFINITY : 0.0;
        total += term;
    }
    return total / (double)L;
}

/* ------------------------------------------------------------------------------------------ */
/* The comparison signal's chunk score (Sec. 4.3; appendix): the write size averaged over the  */
/* heads, the gated-delta layers and the chunk's T tokens, i.e. the sum of all per-(layer,      */
/* head, token) write sizes over L * Hv * T.  T = 0 gives 0.                                    */
/* ------------------------------------------------------------------------------------------ */
double oracle_write_norm_score(int L, int Hv, int T, const double* wnorm)
{
    if (T <= 0) return 0.0;
    double total = 0.0;
    for (size_t i = 0; i < (size_t)L * Hv; ++i) total += wnorm[i];
    return total / ((double)L * Hv * T);
}

/* ------------------------------------------------------------------------------------------ */
/* Retain selection (Sec. 3.3; Alg. 1, eviction branch).                                        */
/*                                                                                              */
/* Inputs: cache length T (slots in stream order), per-slot arrival chunk tok_chunk[T], and the */
/* stored chunk scores (one score per chunk, shared by all of its tokens, Sec. 3.3).            */
/* If T <= M every slot is kept.  Otherwise:                                                    */
/*   sink = slots [0, n_s), window = slots [T - n_w, T)   (always kept)                         */
/*   candidates = the remaining slots, R = M - n_s - n_w  (remaining capacity)                  */
/*   N equal temporal spans over the candidates' arrival chunks [c_lo, c_hi]:                   */
/*       bucket(i) = floor((a_i - c_lo) * N / (c_hi - c_lo + 1))                                */
/*   quota q = floor(R / N); each span keeps its top min(q, |span|) candidates by score;        */
/*   the unused capacity R - (kept so far) goes to the highest-scoring remaining candidates.   */
/* Ranking key: higher score first, ties broken by the lower slot (earlier arrival first).      */
/* Scores are compared as float32 under the IEEE-754 total order (the paper computes all scores */
/* in float32), so -0 < +0 and +inf ranks above every finite score.                              */
/* Output: retain_idx[0..n) ascending, *n_retained = n = min(T, M), mask[T] (optional).         */
/* N = 0 (the paper's "no bucketing") is read as one span.                                      */
/* ------------------------------------------------------------------------------------------ */
static uint32_t total_order_key(float s)
{
    uint32_t b;
    memcpy(&b, &s, sizeof b);
    return (b & 0x80000000u) ? ~b : (b | 0x80000000u);
}

typedef struct { uint32_t score_key; int32_t slot; } ranked_slot;

static int ranked_cmp(const void* pa, const void* pb)
{
    const ranked_slot* a = (const ranked_slot*)pa;
    const ranked_slot* b = (const ranked_slot*)pb;
    if (a->score_key != b->score_key) return (a->score_key > b->score_key) ? -1 : 1; /* score desc */
    return (a->slot < b->slot) ? -1 : (a->slot > b->slot ? 1 : 0);                 /* slot asc */
}

int oracle_select_retain(int M, int n_sink, int n_window, int n_buckets,
                         int T, int n_chunks, const int32_t* tok_chunk, const float* chunk_scores,
                         int32_t* retain_idx, int32_t* n_retained, uint8_t* mask)
{
    if (M < 1 || n_sink < 0 || n_window < 0 || n_buckets < 0 || T < 0) return ORACLE_BAD_ARG;
    if ((long long)M < (long long)n_sink + n_window + 1) return ORACLE_BAD_ARG;
    if (!retain_idx || !n_retained || (T > 0 && (!tok_chunk || !chunk_scores))) return ORACLE_BAD_ARG;
    for (int i = 0; i < T; ++i)
        if (tok_chunk[i] < 0 || tok_chunk[i] >= n_chunks) return ORACLE_BAD_ARG;
    const int N = n_buckets < 1 ? 1 : n_buckets;

    uint8_t* keep = (uint8_t*)calloc((size_t)(T > 0 ? T : 1), 1);
    if (!keep) return ORACLE_NO_MEMORY;

    if (T <= M) {
        for (int i = 0; i < T; ++i) keep[i] = 1;
    } else {
        const int cand_lo = n_sink, cand_hi = T - n_window; /* candidates are [cand_lo, cand_hi) */
        for (int i = 0; i < n_sink; ++i) keep[i] = 1;
        for (int i = cand_hi; i < T; ++i) keep[i] = 1;
        const int R = M - n_sink - n_window;
        int c_lo = tok_chunk[cand_lo], c_hi = tok_chunk[cand_lo];
        for (int i = cand_lo; i < cand_hi; ++i) {
            if (tok_chunk[i] < c_lo) c_lo = tok_chunk[i];
            if (tok_chunk[i] > c_hi) c_hi = tok_chunk[i];
        }
        const long long span = (long long)c_hi - c_lo + 1;
        const int quota = R / N;
        const int n_cand = cand_hi - cand_lo;
        ranked_slot* list = (ranked_slot*)malloc(sizeof(ranked_slot) * (size_t)n_cand);
        if (!list) { free(keep); return ORACLE_NO_MEMORY; }
        int kept = 0;
        /* phase 1: per-span quota, best first */
        for (int j = 0; j < N; ++j) {
            int m = 0;
            for (int i = cand_lo; i < cand_hi; ++i) {
                const long long b = ((long long)(tok_chunk[i] - c_lo) * N) / span;
                if (b == j) {
                    list[m].score_key = total_order_key(chunk_scores[tok_chunk[i]]);
                    list[m].slot = i;
                    ++m;
                }
            }
            qsort(list, (size_t)m, sizeof(ranked_slot), ranked_cmp);
            const int take = m < quota ? m : quota;
            for (int r = 0; r < take; ++r) keep[list[r].slot] = 1;
            kept += take;
        }
        /* phase 2: fill the unused capacity with the best remaining candidates */
        int m = 0;
        for (int i = cand_lo; i < cand_hi; ++i)
            if (!keep[i]) {
                list[m].score_key = total_order_key(chunk_scores[tok_chunk[i]]);
                list[m].slot = i;
                ++m;
            }
        qsort(list, (size_t)m, sizeof(ranked_slot), ranked_cmp);
        const int fill = R - kept;
        for (int r = 0; r < fill && r < m; ++r) keep[list[r].slot] = 1;
        free(list);
    }
    int n = 0;
    for (int i = 0; i < T; ++i) {
        if (keep[i]) retain_idx[n++] = i;
        if (mask) mask[i] = keep[i];
    }
    *n_retained = n;
    free(keep);
    return ORACLE_OK;
}

/* ------------------------------------------------------------------------------------------ */
/* Cache-internal token signals of the controlled comparison (Sec. 4.3 and the appendix table   */
/* of retention signals): the key-norm signal scores a cached token by -||k||_2 and the         */
/* value-norm signal by ||v||_2, per KV head and per token.  Row r of rows[n_rows][D] gets       */
/*     out[r] = sign * sqrt(sum_i rows[r][i]^2),   sign = -1 (negate != 0) or +1.               */
/* ------------------------------------------------------------------------------------------ */
int oracle_row_norm_scores(int n_rows, int D, const float* rows, int negate, double* out)
{
    if (n_rows < 0 || D < 1 || (n_rows > 0 && (!rows || !out))) return ORACLE_BAD_ARG;
    for (int r = 0; r < n_rows; ++r) {
        double s = 0.0;
        for (int i = 0; i < D; ++i) {
            const double x = rows[(size_t)r * D + i];
            s += x * x;
        }
        out[r] = negate ? -sqrt(s) : sqrt(s);
    }
    return ORACLE_OK;
}

/* ------------------------------------------------------------------------------------------ */
/* Retain selection with one score per token (the token-granular signals of Sec. 4.3, ranked  */
/* under the shared policy of Sec. 3.3: the same sink, window, temporal spans, quota and fill  */
/* as oracle_select_retain above).  The only difference: slot i is ranked by tok_scores[i]     */
/* instead of the score of its chunk.  Spans still split the candidates' arrival chunks.        */
/* Ranking key: higher score first (float32 total order), ties to the lower slot.              */
/* ------------------------------------------------------------------------------------------ */
int oracle_select_retain_tokens(int M, int n_sink, int n_window, int n_buckets, int T,
                                const int32_t* tok_chunk, const float* tok_scores,
                                int32_t* retain_idx, int32_t* n_retained, uint8_t* mask)
{
    if (M < 1 || n_sink < 0 || n_window < 0 || n_buckets < 0 || T < 0) return ORACLE_BAD_ARG;
    if ((long long)M < (long long)n_sink + n_window + 1) return ORACLE_BAD_ARG;
    if (!retain_idx || !n_retained || (T > 0 && (!tok_chunk || !tok_scores))) return ORACLE_BAD_ARG;
    for (int i = 0; i < T; ++i)
        if (tok_chunk[i] < 0) return ORACLE_BAD_ARG;
    const int N = n_buckets < 1 ? 1 : n_buckets;

    uint8_t* keep = (uint8_t*)calloc((size_t)(T > 0 ? T : 1), 1);
    if (!keep) return ORACLE_NO_MEMORY;

    if (T <= M) {
        for (int i = 0; i < T; ++i) keep[i] = 1;
    } else {
        const int cand_lo = n_sink, cand_hi = T - n_window;
        for (int i = 0; i < n_sink; ++i) keep[i] = 1;
        for (int i = cand_hi; i < T; ++i) keep[i] = 1;
        const int R = M - n_sink - n_window;
        int c_lo = tok_chunk[cand_lo], c_hi = tok_chunk[cand_lo];
        for (int i = cand_lo; i < cand_hi; ++i) {
            if (tok_chunk[i] < c_lo) c_lo = tok_chunk[i];
            if (tok_chunk[i] > c_hi) c_hi = tok_chunk[i];
        }
        const long long span = (long long)c_hi - c_lo + 1;
        const int quota = R / N;
        const int n_cand = cand_hi - cand_lo;
        ranked_slot* list = (ranked_slot*)malloc(sizeof(ranked_slot) * (size_t)n_cand);
        if (!list) { free(keep); return ORACLE_NO_MEMORY; }
        int kept = 0;
        /* phase 1: per-span quota, best tokens first */
        for (int j = 0; j < N; ++j) {
            int m = 0;
            for (int i = cand_lo; i < cand_hi; ++i) {
                const long long b = ((long long)(tok_chunk[i] - c_lo) * N) / span;
                if (b == j) {
                    list[m].score_key = total_order_key(tok_scores[i]);
                    list[m].slot = i;
                    ++m;
                }
            }
            qsort(list, (size_t)m, sizeof(ranked_slot), ranked_cmp);
            const int take = m < quota ? m : quota;
            for (int r = 0; r < take; ++r) keep[list[r].slot] = 1;
            kept += take;
        }
        /* phase 2: the unused capacity goes to the best remaining tokens of any span */
        int m = 0;
        for (int i = cand_lo; i < cand_hi; ++i)
            if (!keep[i]) {
                list[m].score_key = total_order_key(tok_scores[i]);
                list[m].slot = i;
                ++m;
            }
        qsort(list, (size_t)m, sizeof(ranked_slot), ranked_cmp);
        const int fill = R - kept;
        for (int r = 0; r < fill && r < m; ++r) keep[list[r].slot] = 1;
        free(list);
    }
    int n = 0;
    for (int i = 0; i < T; ++i) {
        if (keep[i]) retain_idx[n++] = i;
        if (mask) mask[i] = keep[i];
    }
    *n_retained = n;
    free(keep);
    return ORACLE_OK;
}

/* ------------------------------------------------------------------------------------------ */
/* KV compaction (Alg. 1, "KV <- KV[I_sink u I_DeltaS u I_window]"; Sec. 3.3: survivors keep    */
/* their original position indices).  Out-of-place gather of fixed-size rows, applied to every */
/* plane independently (each full-attention layer, K and V, each KV head):                      */
/*     out[p][j] = in[p][retain_idx[j]]   for j <  n_retained                                  */
/*     out[p][j] = in[p][j]               for j >= n_retained  (rows past the end untouched)    */
/* Planes have `capacity` rows of row_bytes bytes; only the first `cache_len` rows are valid.   */
/* The same call gathers the per-slot metadata (tok_chunk, tok_pos) as 4-byte rows.             */
/* ------------------------------------------------------------------------------------------ */
int oracle_compact_rows(int n_planes, int capacity, int row_bytes, int cache_len,
                        const uint8_t* in, uint8_t* out, const int32_t* retain_idx, int n_retained)
{
    if (n_planes < 0 || capacity < 0 || row_bytes < 1 || cache_len < 0 || cache_len > capacity) return ORACLE_BAD_ARG;
    if (n_retained < 0 || n_retained > cache_len) return ORACLE_BAD_ARG;
    for (int j = 0; j < n_retained; ++j)
        if (retain_idx[j] < 0 || retain_idx[j] >= cache_len) return ORACLE_BAD_ARG;
    const size_t plane = (size_t)capacity * row_bytes;
    memcpy(out, in, plane * (size_t)n_planes);
    for (int p = 0; p < n_planes; ++p)
        for (int j = 0; j < n_retained; ++j)
            memcpy(out + p * plane + (size_t)j * row_bytes,
                   in + p * plane + (size_t)retain_idx[j] * row_bytes, (size_t)row_bytes);
    return ORACLE_OK;
}
