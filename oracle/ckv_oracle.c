/*
 * ckv_oracle.c -- TEST INFRASTRUCTURE ONLY.
 *
 * A plain, slow, fp64 CPU statement of what CompressKV's prefill-time KV-cache compression step
 * computes (arxiv 2508.02401, Sec. 3.3, token selection by the semantic retrieval heads,
 * with the attention of Eq. 2 and the pooling hyper-parameters of App. A).  It exists to
 * check the CUDA library and is only ever loaded by the tests, by the package's smoke check
 * and by the benchmark's CPU-baseline leg.  It shares no code, header, table or helper with
 * the CUDA library.
 *
 * Everything is written out the obvious way: explicit loops, one value at a time, fp64
 * accumulation, a library sort for the selection.  Inputs are bfloat16 bit patterns (uint16),
 * widened exactly to double.
 *
 * Readings of the paper where it is silent or ambiguous (each one is listed with its reason in
 * the project's design notes):
 *   (i)   logits are scaled by 1/sqrt(d) (standard attention; Eq. 2 prints no scale);
 *   (ii)  window row r is the query at position P + r (P = L - w) and, as in the model's causal
 *         prefill attention, sees keys 0..P+r; its softmax runs over exactly those keys;
 *   (iii) pooling is 1-D, stride 1, same length, over the candidate positions [0, P) only,
 *         padding kernel/2 on each side; max pooling ignores padded cells, average pooling
 *         counts them as zeros and always divides by the kernel size;
 *   (iv)  both head orders are provided: pool each selected head then sum (the order of
 *         Sec. 3.3) or sum the selected heads then pool;
 *   (v)   heads are summed, not averaged (a positive rescale; the ranking is identical);
 *   (vi)  one index set per KV head, from the selected heads of its GQA group (scope 0); or,
 *         as Sec. 3.3 states it, one index set per layer from all of the layer's selected
 *         heads, shared by every KV head (scope 1);
 *   (vii) the budget B counts the window: k = B - w candidates are kept; if L <= B every
 *         position is kept;
 *   (viii) ties in the selection go to the lower position;
 *   (ix)  kept positions are returned in ascending order (the window positions come last);
 *   (x)   query head h belongs to KV group h / (H_q / H_kv).
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>
#ifdef _OPENMP
#include <omp.h>
#endif

#define ORACLE_OK 0
#define ORACLE_BAD_ARG 1
#define ORACLE_NO_MEMORY 2

static double widen_bf16(uint16_t bits) {
    uint32_t u = (uint32_t)bits << 16;
    float f;
    memcpy(&f, &u, sizeof f);
    return (double)f;
}

/*
 * Window attention of one query head over one sequence (Eq. 2; Sec. 3.3 adds up the
 * window rows' attention per key).
 *
 *   q: w rows of d values, row r is the query at sequence position P + r, P = L - w;
 *      consecutive rows are q_row_stride elements apart.
 *   k: L rows of d values, consecutive rows k_row_stride elements apart.
 *   a[j]    (j in [0, L)) = sum over rows r that see key j of p_{r,j}
 *   lse[r]  = log sum_{j <= P+r} exp(s_{r,j}),  s_{r,j} = scale * q_r . k_j
 *             (NaN for a row whose query position is negative, i.e. L < w)
 *   mass[r] = sum_{j >= P} p_{r,j}   (the row's attention on the window keys)
 */
int ckv_oracle_window_scores(int L, int w, int d, double scale,
                             const uint16_t* q, long q_row_stride,
                             const uint16_t* k, long k_row_stride,
                             double* a, double* lse, double* mass) {
    if (L < 0 || w < 1 || d < 1) return ORACLE_BAD_ARG;
    int P = L - w;
    for (int j = 0; j < L; ++j) a[j] = 0.0;
    double* s = (double*)malloc(sizeof(double) * (size_t)(L > 0 ? L : 1));
    if (!s) return ORACLE_NO_MEMORY;
    for (int r = 0; r < w; ++r) {
        int qpos = P + r;
        if (qpos < 0) {
            if (lse) lse[r] = NAN;
            if (mass) mass[r] = 0.0;
            continue;
        }
        const uint16_t* qr = q + (long)r * q_row_stride;
        double mx = -INFINITY;
        for (int j = 0; j <= qpos; ++j) {
            const uint16_t* kj = k + (long)j * k_row_stride;
            double dot = 0.0;
            for (int c = 0; c < d; ++c) dot += widen_bf16(qr[c]) * widen_bf16(kj[c]);
            s[j] = scale * dot;
            if (s[j] > mx) mx = s[j];
        }
        double sum = 0.0;
        for (int j = 0; j <= qpos; ++j) sum += exp(s[j] - mx);
        double row_lse = mx + log(sum);
        double row_mass = 0.0;
        for (int j = 0; j <= qpos; ++j) {
            double p = exp(s[j] - row_lse);
            a[j] += p;
            if (j >= P) row_mass += p;
        }
        if (lse) lse[r] = row_lse;
        if (mass) mass[r] = row_mass;
    }
    free(s);
    return ORACLE_OK;
}

/*
 * The same window scores with the rows' normalisers given (lse_in[r], natural log), as a
 * prefill attention kernel returns them for its query rows (Sec. 3.3 with Eq. 2):
 *   a[j] = sum over rows r that see key j of exp(s_{r,j} - lse_in[r]).
 * Rows whose query position is negative (L < w) contribute nothing and lse_in[r] is not read.
 */
int ckv_oracle_window_scores_lse(int L, int w, int d, double scale,
                                 const uint16_t* q, long q_row_stride,
                                 const uint16_t* k, long k_row_stride,
                                 const double* lse_in, double* a) {
    if (L < 0 || w < 1 || d < 1 || !lse_in) return ORACLE_BAD_ARG;
    int P = L - w;
    for (int j = 0; j < L; ++j) a[j] = 0.0;
    for (int r = 0; r < w; ++r) {
        int qpos = P + r;
        if (qpos < 0) continue;
        const uint16_t* qr = q + (long)r * q_row_stride;
        for (int j = 0; j <= qpos; ++j) {
            const uint16_t* kj = k + (long)j * k_row_stride;
            double dot = 0.0;
            for (int c = 0; c < d; ++c) dot += widen_bf16(qr[c]) * widen_bf16(kj[c]);
            a[j] += exp(scale * dot - lse_in[r]);
        }
    }
    return ORACLE_OK;
}

/*
 * 1-D pooling along the token axis (Sec. 3.3; App. A uses kernel 5 with average pooling).
 * Stride 1, output length n, window [j - kernel/2, j + kernel/2] clipped to [0, n).
 *   type 0 (max): maximum over the clipped window (padded cells ignored);
 *   type 1 (avg): sum over the clipped window divided by kernel (zero padding counted).
 */
int ckv_oracle_pool(const double* x, int n, int kernel, int type, double* y) {
    if (n < 0 || kernel < 1 || (kernel % 2) == 0 || (type != 0 && type != 1)) return ORACLE_BAD_ARG;
    int half = kernel / 2;
    for (int j = 0; j < n; ++j) {
        int lo = j - half < 0 ? 0 : j - half;
        int hi = j + half > n - 1 ? n - 1 : j + half;
        if (type == 0) {
            double m = x[lo];
            for (int t = lo + 1; t <= hi; ++t)
                if (x[t] > m) m = x[t];
            y[j] = m;
        } else {
            double sum = 0.0;
            for (int t = lo; t <= hi; ++t) sum += x[t];
            y[j] = sum / (double)kernel;
        }
    }
    return ORACLE_OK;
}

typedef struct {
    double value;
    int32_t pos;
} scored_pos;

static int by_value_desc_then_pos(const void* pa, const void* pb) {
    const scored_pos* a = (const scored_pos*)pa;
    const scored_pos* b = (const scored_pos*)pb;
    if (a->value > b->value) return -1;
    if (a->value < b->value) return 1;
    return (a->pos > b->pos) - (a->pos < b->pos);
}

static int by_int_asc(const void* pa, const void* pb) {
    int32_t a = *(const int32_t*)pa, b = *(const int32_t*)pb;
    return (a > b) - (a < b);
}

/*
 * Top-N selection (Sec. 3.3): the k positions of c[0..P) with the largest values, ties to the
 * lower position, written to out[0..k) in ascending order.
 */
int ckv_oracle_topk(const double* c, int P, int k, int32_t* out) {
    if (P < 0 || k < 0 || k > P) return ORACLE_BAD_ARG;
    if (k == 0) return ORACLE_OK;
    scored_pos* v = (scored_pos*)malloc(sizeof(scored_pos) * (size_t)P);
    if (!v) return ORACLE_NO_MEMORY;
    for (int j = 0; j < P; ++j) {
        v[j].value = c[j];
        v[j].pos = j;
    }
    qsort(v, (size_t)P, sizeof(scored_pos), by_value_desc_then_pos);
    for (int i = 0; i < k; ++i) out[i] = v[i].pos;
    qsort(out, (size_t)k, sizeof(int32_t), by_int_asc);
    free(v);
    return ORACLE_OK;
}

/* Tokens kept per KV head for each sequence: min(B, L_s) (reading vii). cu_keep[S+1]. */
int ckv_oracle_keep_lengths(int S, const int32_t* cu_seqlens, int budget, int32_t* cu_keep) {
    if (S < 0 || budget < 0) return ORACLE_BAD_ARG;
    cu_keep[0] = 0;
    for (int s = 0; s < S; ++s) {
        int L = cu_seqlens[s + 1] - cu_seqlens[s];
        if (L < 0) return ORACLE_BAD_ARG;
        cu_keep[s + 1] = cu_keep[s] + (L < budget ? L : budget);
    }
    return ORACLE_OK;
}

/*
 * One layer of the compression step over a varlen batch (Sec. 3.3, Fig. 3).
 *
 * Inputs (bf16 bits, packed row-major):
 *   q_win [S, w, Hq, d]   the last w query rows of each sequence
 *   k, v  [T, Hkv, d]     T = cu_seqlens[S]
 *   head_mask [Hq]        1 = selected (semantic retrieval) head of this layer
 * Outputs (any of scores/pooled/idx/k_out/v_out may be NULL to skip it):
 *   scores [n_sel, T]     a_h for each selected head h (rows in ascending h), all positions
 *   pooled [Hkv, T]       c_g on the candidate positions [0, P_s), 0 elsewhere
 *   cu_keep [S+1]         prefix sums of min(B, L_s)
 *   idx   [Hkv, T_keep]   kept sequence-local positions, ascending, per (KV head, sequence)
 *   k_out, v_out [T_keep, Hkv, d]  the kept rows
 * group_filter (optional, [Hkv]): when given, only groups with a non-zero entry are computed.
 */
/*
 * One layer of the step (Sec. 3.3).  scope 0: a vector, a selection and an index set per KV
 * head g from the selected heads of group g.  scope 1: one vector and one selection per
 * sequence from every selected head of the layer (each head against its own group's keys);
 * the index set is repeated for every KV head and each KV head's rows are gathered with it.
 * pooled has Hkv rows (scope 0) or 1 row (scope 1); idx and the outputs have Hkv rows.
 * lse_in (optional): the window rows' normalisers, lse_in[h * lse_head_stride + s * w + r]
 * (natural log), used instead of computing them (ckv_oracle_window_scores_lse).
 */
int ckv_oracle_compress_layer(int S, const int32_t* cu_seqlens, int Hq, int Hkv, int d, int w,
                              double scale, const uint8_t* head_mask, int budget,
                              int pool_kernel, int pool_type, int head_order, int scope,
                              const uint16_t* q_win, const uint16_t* k, const uint16_t* v,
                              const double* lse_in, long lse_head_stride,
                              double* scores, double* pooled, int32_t* cu_keep, int32_t* idx,
                              uint16_t* k_out, uint16_t* v_out, const uint8_t* group_filter,
                              int num_threads) {
    if (S < 0 || Hq < 1 || Hkv < 1 || Hq % Hkv != 0 || d < 1 || w < 1 || budget < w ||
        pool_kernel < 1 || pool_kernel % 2 == 0 || (pool_type != 0 && pool_type != 1) ||
        (head_order != 0 && head_order != 1) || (scope != 0 && scope != 1) ||
        (scope == 1 && group_filter))
        return ORACLE_BAD_ARG;
    const int n_vec = scope == 0 ? Hkv : 1; /* selections per sequence */
    const int G = Hq / Hkv;
    const int T = cu_seqlens[S];
    int32_t* keep = (int32_t*)malloc(sizeof(int32_t) * (size_t)(S + 1));
    int* sel_row = (int*)malloc(sizeof(int) * (size_t)Hq); /* row of head h in scores, or -1 */
    if (!keep || !sel_row) {
        free(keep);
        free(sel_row);
        return ORACLE_NO_MEMORY;
    }
    int rc = ckv_oracle_keep_lengths(S, cu_seqlens, budget, keep);
    if (rc) {
        free(keep);
        free(sel_row);
        return rc;
    }
    if (cu_keep) memcpy(cu_keep, keep, sizeof(int32_t) * (size_t)(S + 1));
    const int Tk = keep[S];
    int n_sel = 0;
    for (int h = 0; h < Hq; ++h) sel_row[h] = head_mask[h] ? n_sel++ : -1;
    for (int g = 0; g < n_vec; ++g) {
        int any = 0;
        const int h0 = scope == 0 ? g * G : 0, h1 = scope == 0 ? (g + 1) * G : Hq;
        for (int h = h0; h < h1; ++h) any |= head_mask[h] != 0;
        if (!any) {
            free(keep);
            free(sel_row);
            return ORACLE_BAD_ARG; /* every selection needs a selected head */
        }
    }
    int failed = 0;
#ifdef _OPENMP
    if (num_threads > 0) omp_set_num_threads(num_threads);
#pragma omp parallel for schedule(dynamic, 1) reduction(| : failed)
#endif
    for (int unit = 0; unit < S * n_vec; ++unit) {
        const int s = unit / n_vec, g = unit % n_vec; /* g: the KV head, or 0 (scope 1) */
        if (group_filter && !group_filter[g]) continue;
        const int t0 = cu_seqlens[s];
        const int L = cu_seqlens[s + 1] - t0;
        const int P = L - w;
        const int Pc = P > 0 ? P : 0;
        double* a = (double*)malloc(sizeof(double) * (size_t)(L > 0 ? L : 1));
        double* acc = (double*)calloc((size_t)(L > 0 ? L : 1), sizeof(double));
        double* tmp = (double*)malloc(sizeof(double) * (size_t)(L > 0 ? L : 1));
        double* lse = (double*)malloc(sizeof(double) * (size_t)w);
        double* mass = (double*)malloc(sizeof(double) * (size_t)w);
        if (!a || !acc || !tmp || !lse || !mass) {
            failed |= 1;
            free(a); free(acc); free(tmp); free(lse); free(mass);
            continue;
        }
        /* steps 1-3: per selected head, window attention summed over the window rows, then
         * pooled and summed over heads (head_order 0) or summed and then pooled (1) */
        const int h0 = scope == 0 ? g * G : 0, h1 = scope == 0 ? (g + 1) * G : Hq;
        for (int h = h0; h < h1; ++h) {
            if (!head_mask[h]) continue;
            const uint16_t* qh = q_win + ((long)s * w * Hq + h) * d;
            const uint16_t* kg = k + ((long)t0 * Hkv + h / G) * d; /* the head's own KV group */
            const int ws_rc =
                lse_in ? ckv_oracle_window_scores_lse(L, w, d, scale, qh, (long)Hq * d, kg,
                                                      (long)Hkv * d,
                                                      lse_in + (long)h * lse_head_stride + (long)s * w, a)
                       : ckv_oracle_window_scores(L, w, d, scale, qh, (long)Hq * d, kg, (long)Hkv * d,
                                                  a, lse, mass);
            if (ws_rc) {
                failed |= 1;
                continue;
            }
            if (scores)
                for (int j = 0; j < L; ++j) scores[(long)sel_row[h] * T + t0 + j] = a[j];
            if (head_order == 0) {
                ckv_oracle_pool(a, Pc, pool_kernel, pool_type, tmp);
                for (int j = 0; j < Pc; ++j) acc[j] += tmp[j];
            } else {
                for (int j = 0; j < Pc; ++j) acc[j] += a[j];
            }
        }
        if (head_order == 1) {
            ckv_oracle_pool(acc, Pc, pool_kernel, pool_type, tmp);
            memcpy(acc, tmp, sizeof(double) * (size_t)Pc);
        }
        if (pooled)
            for (int j = 0; j < L; ++j) pooled[(long)g * T + t0 + j] = j < Pc ? acc[j] : 0.0;
        /* step 4: top-(B - w) candidates plus the w window positions, or everything if L <= B */
        const int ks = keep[s], kn = keep[s + 1] - keep[s];
        int32_t* out = (int32_t*)malloc(sizeof(int32_t) * (size_t)(kn > 0 ? kn : 1));
        if (!out) {
            failed |= 1;
        } else {
            if (L <= budget) {
                for (int i = 0; i < L; ++i) out[i] = i;
            } else {
                int kc = budget - w;
                if (ckv_oracle_topk(acc, P, kc, out)) failed |= 1;
                for (int i = 0; i < w; ++i) out[kc + i] = P + i;
            }
            /* step 5: the kept K/V rows, in position order, for the KV head (scope 0) or for
             * every KV head (scope 1) */
            const int kv0 = scope == 0 ? g : 0, kv1 = scope == 0 ? g + 1 : Hkv;
            for (int kv = kv0; kv < kv1; ++kv)
                for (int i = 0; i < kn; ++i) {
                    if (idx) idx[(long)kv * Tk + ks + i] = out[i];
                    long src = ((long)(t0 + out[i]) * Hkv + kv) * d;
                    long dst = ((long)(ks + i) * Hkv + kv) * d;
                    if (k_out) memcpy(k_out + dst, k + src, sizeof(uint16_t) * (size_t)d);
                    if (v_out) memcpy(v_out + dst, v + src, sizeof(uint16_t) * (size_t)d);
                }
            free(out);
        }
        free(a); free(acc); free(tmp); free(lse); free(mass);
    }
    free(keep);
    free(sel_row);
    return failed ? ORACLE_NO_MEMORY : ORACLE_OK;
}

/*
 * Semantic Retrieval Score (Sec. 3.2, Eq. 5), added into srs[Hq] for the selected heads:
 *   srs[h] += sum over decode steps t with in_answer[s*w + t] of sum_{j in [a0, a1)} a^h_{t,j}
 * per sequence s, where a^h_{t,j} is head h's attention of decode step t over keys
 * 0..L_s-w+t (the context and the generated tokens up to itself; Eq. 2 with scale) and
 * [a0, a1) = span[2s], span[2s+1] is the answer span.  q_dec [S, w, Hq, d], k [T, Hkv, d].
 */
int ckv_oracle_srs(int S, const int32_t* cu_seqlens, int Hq, int Hkv, int d, int w, double scale,
                   const uint8_t* head_mask, const uint16_t* q_dec, const uint16_t* k,
                   const uint8_t* in_answer, const int32_t* span, double* srs) {
    if (S < 0 || Hq < 1 || Hkv < 1 || Hq % Hkv != 0 || d < 1 || w < 1) return ORACLE_BAD_ARG;
    const int G = Hq / Hkv;
    for (int s = 0; s < S; ++s) {
        const int t0 = cu_seqlens[s], L = cu_seqlens[s + 1] - t0;
        const int a0 = span[2 * s], a1 = span[2 * s + 1];
        if (a0 < 0 || a1 < a0 || a1 > L) return ORACLE_BAD_ARG;
        double* logit = (double*)malloc(sizeof(double) * (size_t)(L > 0 ? L : 1));
        if (!logit) return ORACLE_NO_MEMORY;
        for (int h = 0; h < Hq; ++h) {
            if (!head_mask[h]) continue;
            for (int t = 0; t < w; ++t) {
                if (!in_answer[s * w + t]) continue;
                const int last = L - w + t; /* the step's own position */
                if (last < 0) continue;
                const uint16_t* qt = q_dec + (((long)s * w + t) * Hq + h) * d;
                double mx = -INFINITY;
                for (int j = 0; j <= last; ++j) {
                    const uint16_t* kj = k + ((long)(t0 + j) * Hkv + h / G) * d;
                    double dot = 0.0;
                    for (int c = 0; c < d; ++c) dot += widen_bf16(qt[c]) * widen_bf16(kj[c]);
                    logit[j] = scale * dot;
                    if (logit[j] > mx) mx = logit[j];
                }
                double z = 0.0;
                for (int j = 0; j <= last; ++j) z += exp(logit[j] - mx);
                double on_span = 0.0;
                for (int j = a0; j < a1 && j <= last; ++j) on_span += exp(logit[j] - mx);
                srs[h] += on_span / z;
            }
        }
        free(logit);
    }
    return ORACLE_OK;
}

/* Number of threads an OpenMP region of this library uses when asked for n (0 = default). */
int ckv_oracle_threads(int n) {
#ifdef _OPENMP
    if (n > 0) return n;
    return omp_get_max_threads();
#else
    (void)n;
    return 1;
#endif
}
