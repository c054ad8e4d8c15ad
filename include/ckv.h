/*
 * ckv.h -- C ABI of libckv, a GB300 (sm_103a) implementation of CompressKV's prefill-time
 * KV-cache compression step (arxiv 2508.02401, Sec. 3.3 and Fig. 3, token selection by the
 * semantic retrieval heads; attention as in Eq. 2; pooling hyper-parameters from App. A).
 *
 * For one transformer layer and every GQA KV head g, the step
 *   1. scores every prefix token j by the attention that the observation window (the last w
 *      query rows) of the layer's selected heads in group g pays to it:
 *        a_h[j] = sum_r softmax_j(scale * q_{h,r} . k_{g,j}),  row r sees keys j <= L - w + r;
 *   2. smooths a_h along the token axis with a 1-D pool and combines the selected heads;
 *   3. keeps the top (B_l - w) candidate positions j < L - w (B_l = the layer's budget) plus
 *      the w window positions, in ascending order (every position when L <= B_l);
 *   4. gathers the kept K/V rows into a compacted, position-ordered cache.
 *
 * Conventions shared by every entry point
 *   - Pointers named *_dev and all tensor arguments are DEVICE memory of the current CUDA
 *     device; pointers named *_host and the config's head mask / budgets are HOST memory.
 *   - Tensors are bfloat16 unless stated; head_dim is 128.  Layouts, row-major:
 *       q_win  [S, w, H_q, 128]       the last w query rows of every sequence (packed)
 *       k, v   [T, H_kv, 128]         varlen-packed by cu_seqlens; element (t, g, c) lives at
 *                                     t*tok_stride + g*head_stride + c (strides in elements,
 *                                     0 = packed: tok_stride = H_kv*128, head_stride = 128)
 *       scores [n_sel, T]   fp32      one row per selected head of the layer, in ascending
 *                                     query-head order (so grouped by KV head)
 *       pooled [n_vec, T]   fp32      combined, pooled scores on candidate positions; 0 at the
 *                                     window positions; n_vec = H_kv (CKV_SCOPE_KV_HEAD) or 1
 *                                     (CKV_SCOPE_LAYER)
 *       idx    [H_kv, T_keep] int32   kept sequence-local positions; the positions of sequence
 *                                     s for head g are idx[g*T_keep + cu_keep[s] ...] (the same
 *                                     for every g with CKV_SCOPE_LAYER)
 *       k_out, v_out [T_keep, H_kv, 128]  packed
 *     with T = cu_seqlens[S], T_keep = sum_s min(B_l, L_s).
 *   - The caller owns every buffer.  The library allocates no device or host memory during a
 *     call and keeps no per-call state; all work is enqueued asynchronously on `stream`
 *     (NULL = the legacy default stream).  Only ckv_read_device_status synchronises.
 *   - Argument errors are detected on the host before anything is enqueued and leave every
 *     output untouched.  No entry point aborts, exits or throws.  Errors that only the device
 *     can see (cu_seqlens_dev disagreeing with cu_seqlens_host, a kernel wait that timed out)
 *     are recorded in the workspace's status word and reported by ckv_read_device_status.
 *   - Device pointers must be 16-byte aligned, the workspace 256-byte aligned.
 *   - A workspace may be reused by calls that are ordered on one stream; calls that may run
 *     concurrently need separate workspaces.  Zero it once (cudaMemset) before its first use,
 *     and again after a call that returned CKV_ERR_CUDA: the selection keeps a histogram there
 *     that each call leaves zeroed for the next.
 */
#ifndef CKV_H
#define CKV_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

#define CKV_ABI_VERSION 7

#if defined(__GNUC__)
#define CKV_API __attribute__((visibility("default")))
#else
#define CKV_API
#endif

typedef struct CUstream_st* ckv_stream; /* the same type as cudaStream_t */

typedef enum ckv_status {
    CKV_OK = 0,
    CKV_ERR_INVALID_ARG = 1, /* a pointer, size, layout or config field is invalid */
    CKV_ERR_UNSUPPORTED = 2, /* valid, but outside what this build supports (e.g. head_dim) */
    CKV_ERR_WORKSPACE = 3,   /* workspace missing, misaligned or smaller than required */
    CKV_ERR_CUDA = 4,        /* a CUDA runtime call failed; see ckv_last_error_message() */
    CKV_ERR_DEVICE = 5       /* a kernel recorded an error in the workspace status word */
} ckv_status;

/* Which heads' vectors make one selection (Sec. 3.3). */
typedef enum ckv_scope {
    CKV_SCOPE_KV_HEAD = 0, /* one selection per KV head g from the selected heads of group g;
                              each KV head keeps its own positions */
    CKV_SCOPE_LAYER = 1    /* one selection per sequence from every selected head of the layer
                              (the form Sec. 3.3 states); every KV head keeps those positions */
} ckv_scope;

/* Which scoring kernel runs the two passes over the keys (same scores either way). */
typedef enum ckv_score_path {
    CKV_SCORE_AUTO = 0,     /* resident when it fits and N = 32 (see below), otherwise reload */
    CKV_SCORE_RESIDENT = 1, /* each key tile is read and multiplied once; pass 1 keeps its
                               exponentials in tensor memory and pass 2 rescales them.  Needs
                               every sequence's key tiles to fit one round of work items of at
                               most 512 / N tiles (N = 32 or 64 window-row columns of a head
                               batch); CKV_ERR_UNSUPPORTED if not */
    CKV_SCORE_RELOAD = 2    /* pass 2 reads each key tile again (from L2 while it is there) and
                               multiplies it again; no limit on the sequence length */
} ckv_score_path;

typedef enum ckv_pool_type { CKV_POOL_MAX = 0, CKV_POOL_AVG = 1 } ckv_pool_type;

/* How the selected heads of a KV group are combined (Sec. 3.3 pools each head's window sum
 * and then averages the vectors; averaging is replaced by summing, which ranks identically). */
typedef enum ckv_head_order {
    CKV_POOL_THEN_SUM = 0, /* c_g = sum_h pool(a_h)  -- the order of Sec. 3.3 */
    CKV_SUM_THEN_POOL = 1  /* c_g = pool(sum_h a_h) */
} ckv_head_order;

/* Per-model settings.  head_mask and budgets are the paper's per-layer head-selection mask
 * (Sec. 3.3, top Semantic Retrieval Heads per layer, Eq. 5) and per-layer budgets (Sec. 3.4,
 * Algorithm 1); both stay in host memory and are read during each call. */
typedef struct ckv_config {
    int32_t num_layers;
    int32_t num_q_heads;   /* H_q, a multiple of num_kv_heads; at most 256 */
    int32_t num_kv_heads;  /* H_kv; query head h belongs to KV head h / (H_q / H_kv) */
    int32_t head_dim;      /* must be 128 */
    int32_t window;        /* w, observation window rows, 1..64 */
    int32_t pool_kernel;   /* odd, 1..63; 1 = no pooling */
    int32_t pool_type;     /* ckv_pool_type: max ignores padding; avg counts zero padding and
                              divides by pool_kernel */
    int32_t head_order;    /* ckv_head_order */
    int32_t scope;         /* ckv_scope; n_vec = num_kv_heads (CKV_SCOPE_KV_HEAD) or 1
                              (CKV_SCOPE_LAYER) selections per sequence */
    float softmax_scale;   /* scale of q.k; 0 selects 1/sqrt(head_dim) */
    int32_t max_ctas;      /* SMs one call's scoring kernel may occupy; 0 = all.  Callers that
                              run several layers concurrently on different streams give each
                              call a share, so the calls' kernels can be resident together. */
    int32_t score_path;    /* ckv_score_path */
    const uint8_t* head_mask; /* host [num_layers * num_q_heads]; non-zero = selected.  With
                                 CKV_SCOPE_KV_HEAD every KV group of a layer needs at least one
                                 selected head; with CKV_SCOPE_LAYER the layer needs one. */
    const int32_t* budgets;   /* host [num_layers]; kept tokens per KV head, window included,
                                 >= window */
} ckv_config;

/* A varlen batch: sequence s occupies tokens [cu_seqlens[s], cu_seqlens[s+1]). */
typedef struct ckv_batch {
    int32_t num_seqs;               /* S >= 1 */
    const int32_t* cu_seqlens_host; /* host   [S+1], cu[0] = 0, non-decreasing */
    const int32_t* cu_seqlens_dev;  /* device [S+1], the same values */
} ckv_batch;

/* Version of this ABI (CKV_ABI_VERSION of the built library). */
CKV_API int32_t ckv_abi_version(void);

/* Human-readable name of a status code (static storage). */
CKV_API const char* ckv_status_string(ckv_status status);

/* Detail of the last failing call on this host thread (static thread-local storage). */
CKV_API const char* ckv_last_error_message(void);

/* Workspace bytes that every entry point below needs for (cfg, layer, batch).  Host only. */
CKV_API ckv_status ckv_workspace_size(const ckv_config* cfg, int32_t layer, const ckv_batch* batch,
                              size_t* bytes);

/* Host only: cu_keep_host[S+1] = prefix sums of min(B_layer, L_s), and the number of score
 * rows n_sel of the layer (may be NULL). */
CKV_API ckv_status ckv_keep_lengths(const ckv_config* cfg, int32_t layer, const ckv_batch* batch,
                            int32_t* cu_keep_host, int32_t* n_sel);

/* Step 1 (Sec. 3.3, with the attention of Eq. 2; the window rows' probabilities are added):
 * scores[i, t] = a_h[j] for the i-th selected head h of the layer and every token t = cu[s]+j,
 * including window positions (there a_h[j] sums only the rows that see key j).  The softmax of
 * window row r runs over keys 0..L-w+r (causal).  Computed for every sequence of the batch. */
CKV_API ckv_status ckv_score_window(const ckv_config* cfg, int32_t layer, const ckv_batch* batch,
                            const void* q_win, const void* k, int64_t tok_stride,
                            int64_t head_stride, float* scores, void* workspace,
                            size_t workspace_bytes, ckv_stream stream);

/* Step 1 with the window rows' normalisers given (the log-sum-exp that a prefill attention
 * kernel returns per query row): the same scores as ckv_score_window, with lse_{h,r} read
 * instead of computed, so K is read and multiplied once and no CTA waits for another.
 *   lse: device fp32, natural log of sum_{j <= P+r} exp(scale * q_{h,r}.k_j) for query head
 *        h and window row r of sequence s at lse[h * lse_head_stride + s * w + r] (the layout
 *        of a varlen prefill's per-head lse over the window rows); lse_head_stride >= S * w,
 *        0 selects S * w.  Only the selected heads' rows are read, and rows whose query
 *        position is before the sequence start (L < w) are not read.  4-byte aligned.
 * The result is exact for the true lse; any other value scales row r's probabilities by
 * exp(lse_true - lse_given). */
CKV_API ckv_status ckv_score_window_lse(const ckv_config* cfg, int32_t layer,
                                        const ckv_batch* batch, const void* q_win, const void* k,
                                        int64_t tok_stride, int64_t head_stride, const float* lse,
                                        int64_t lse_head_stride, float* scores, void* workspace,
                                        size_t workspace_bytes, ckv_stream stream);

/* Step 2 (Sec. 3.3 token-axis smoothing; App. A sizes): pooled[g, cu[s]+j] for
 * j < L_s - w from the scores of selection g's heads (group g's selected heads, or every
 * selected head of the layer with CKV_SCOPE_LAYER), in cfg->head_order; 0 at window positions.
 * Pooling runs over the candidate range only (window scores never enter it). */
CKV_API ckv_status ckv_pool(const ckv_config* cfg, int32_t layer, const ckv_batch* batch,
                    const float* scores, float* pooled, ckv_stream stream);

/* Step 3 (Sec. 3.3, top-N selection):
 * per (sequence, selection), the B_l - w largest pooled candidates (ties: lower position
 * first) followed by the window positions, ascending; every position when L_s <= B_l.  Writes
 * idx for the KV heads the selection serves (its own, or all of them with CKV_SCOPE_LAYER)
 * and cu_keep_dev[S+1] (device copy of ckv_keep_lengths). */
CKV_API ckv_status ckv_select_topk(const ckv_config* cfg, int32_t layer, const ckv_batch* batch,
                           const float* pooled, int32_t* idx, int32_t* cu_keep_dev,
                           void* workspace, size_t workspace_bytes, ckv_stream stream);

/* Step 4 (Sec. 3.3, the kept tokens' K/V pairs form the new cache): k_out / v_out rows
 * = the k / v rows at idx.  t_keep = cu_keep[S].  Bit copy. */
CKV_API ckv_status ckv_gather_compact(const ckv_config* cfg, const ckv_batch* batch, int32_t t_keep,
                              const void* k, const void* v, int64_t tok_stride,
                              int64_t head_stride, const int32_t* idx,
                              const int32_t* cu_keep_dev, void* k_out, void* v_out,
                              void* workspace, size_t workspace_bytes, ckv_stream stream);

/* Steps 2-4 for one layer, fused (the selection half of ckv_compress_layer): pooling, top-k,
 * compaction and the K/V gather from the scores ckv_score_window (or ckv_score_window_lse)
 * wrote.  Splitting a layer into these two calls lets a caller put each layer's selection on
 * a stream of its own, so that the next layer's scoring need not wait for it.
 *   scores: device fp32 [n_sel, T] as ckv_score_window writes it (row i = the layer's i-th
 *           selected head), 16-byte aligned; read only for sequences with L_s > B_l.
 *   k, v, tok_stride, head_stride, idx, cu_keep_dev, k_out, v_out, pooled_out: as for
 *           ckv_compress_layer.  The workspace may be another call's than the scoring's. */
CKV_API ckv_status ckv_select_compact(const ckv_config* cfg, int32_t layer, const ckv_batch* batch,
                                      const float* scores, const void* k, const void* v,
                                      int64_t tok_stride, int64_t head_stride, int32_t* idx,
                                      int32_t* cu_keep_dev, void* k_out, void* v_out,
                                      float* pooled_out, void* workspace, size_t workspace_bytes,
                                      ckv_stream stream);

/* One layer of a multi-layer call (ckv_score_windows(_lse), ckv_compress_layers(_lse)).  The
 * layers of a call share the config and the batch; each brings its own buffers. */
typedef struct ckv_layer_io {
    int32_t layer;                 /* index into the config's head_mask and budgets */
    const void* q_win;             /* [S, w, H_q, 128] */
    const void* k;                 /* [T, H_kv, 128] with the strides below */
    const void* v;                 /* ckv_compress_layers only; the same strides as k */
    int64_t tok_stride;            /* of k and v, in elements; 0 = packed */
    int64_t head_stride;
    float* scores;                 /* ckv_score_windows(_lse): [n_sel, T] out, as ckv_score_window */
    int32_t* idx;                  /* ckv_compress_layers: outputs as for ckv_compress_layer */
    int32_t* cu_keep_dev;
    void* k_out;
    void* v_out;
    float* pooled_out;             /* may be NULL */
    const float* lse;              /* the _lse calls: the window rows' lse, as for
                                      ckv_score_window_lse (fp32, natural log, [H_q][S*w]) */
    int64_t lse_head_stride;       /* elements between heads; 0 = S*w */
} ckv_layer_io;

/* Workspace bytes for a multi-layer call over io[0..n_layers) (enough for either entry point). */
CKV_API ckv_status ckv_workspace_size_layers(const ckv_config* cfg, int32_t n_layers,
                                             const ckv_layer_io* io, const ckv_batch* batch,
                                             size_t* bytes);

/* Step 1 for several layers at once: for each io[i], what ckv_score_window(cfg, io[i].layer,
 * ...) writes to io[i].scores.  Every layer's two passes run in one persistent launch (one per
 * 32 layers, and per 256 sequences), so the GPU streams one layer's keys while it exchanges
 * another's row statistics; the per-call start and tail are paid once.  Always the two-pass
 * kernel that re-reads K in pass 2 (cfg->score_path is ignored).  cfg->max_ctas caps the CTAs
 * of the launch (0 = all SMs), which leaves the other SMs to work issued on other streams. */
CKV_API ckv_status ckv_score_windows(const ckv_config* cfg, int32_t n_layers,
                                     const ckv_layer_io* io, const ckv_batch* batch,
                                     void* workspace, size_t workspace_bytes, ckv_stream stream);

/* Step 1 for several layers with every layer's window-row lse given (io[i].lse and
 * io[i].lse_head_stride, as for ckv_score_window_lse): for each io[i], what
 * ckv_score_window_lse(cfg, io[i].layer, ...) writes to io[i].scores.  Every layer's single
 * pass over K runs in one persistent launch (one per 32 layers, and per 256 sequences); the CTAs
 * take pieces of the (layer, head batch, sequence) units from a global counter, and no CTA
 * waits for another.  CKV_ERR_INVALID_ARG for a NULL lse or a head stride below S*w; otherwise
 * as ckv_score_windows. */
CKV_API ckv_status ckv_score_windows_lse(const ckv_config* cfg, int32_t n_layers,
                                         const ckv_layer_io* io, const ckv_batch* batch,
                                         void* workspace, size_t workspace_bytes,
                                         ckv_stream stream);

/* Steps 1-4 for several layers: for each io[i], what ckv_compress_layer(cfg, io[i].layer, ...)
 * writes.  The layers are scored as by ckv_score_windows (into the workspace), then every
 * layer's selection runs in one launch (one per 32 layers) on the same stream, each (layer,
 * sequence, selection) by one CTA that keeps a list of the keys that can still be kept in the
 * workspace.  Sequences with L_s at most every layer's budget are copied whole without being
 * scored.  The workspace (ckv_workspace_size_layers) holds, per layer, the scores [n_sel, T]
 * fp32 (and 64 bytes after them, which the selection's TMA view of them may read) and the
 * selection's lists [H_kv, T + 4 S] of 8-byte entries, and per unit of the scoring launch N
 * fp64 row sums and a counter. */
CKV_API ckv_status ckv_compress_layers(const ckv_config* cfg, int32_t n_layers,
                                       const ckv_layer_io* io, const ckv_batch* batch,
                                       void* workspace, size_t workspace_bytes, ckv_stream stream);

/* Steps 1-4 for several layers with every layer's window-row lse given (io[i].lse: the lse a
 * prefill attention kernel returns): for each io[i], what ckv_compress_layer_lse(cfg,
 * io[i].layer, ...) writes.  The layers are scored as by ckv_score_windows_lse (one pass over
 * K, into the workspace), then every layer's selection runs in one launch as in
 * ckv_compress_layers.  The same workspace (ckv_workspace_size_layers).  cfg->score_path is
 * ignored. */
CKV_API ckv_status ckv_compress_layers_lse(const ckv_config* cfg, int32_t n_layers,
                                           const ckv_layer_io* io, const ckv_batch* batch,
                                           void* workspace, size_t workspace_bytes,
                                           ckv_stream stream);

/* Steps 1-4 for one layer.  Sequences with L_s <= B_l are copied whole without being scored.
 * pooled_out may be NULL (then the pooled scores stay in the workspace). */
CKV_API ckv_status ckv_compress_layer(const ckv_config* cfg, int32_t layer, const ckv_batch* batch,
                              const void* q_win, const void* k, const void* v,
                              int64_t tok_stride, int64_t head_stride, int32_t* idx,
                              int32_t* cu_keep_dev, void* k_out, void* v_out, float* pooled_out,
                              void* workspace, size_t workspace_bytes, ckv_stream stream);

/* ckv_compress_layer with the window rows' lse given (layout as in ckv_score_window_lse). */
CKV_API ckv_status ckv_compress_layer_lse(const ckv_config* cfg, int32_t layer,
                                          const ckv_batch* batch, const void* q_win,
                                          const void* k, const void* v, int64_t tok_stride,
                                          int64_t head_stride, const float* lse,
                                          int64_t lse_head_stride, int32_t* idx,
                                          int32_t* cu_keep_dev, void* k_out, void* v_out,
                                          float* pooled_out, void* workspace,
                                          size_t workspace_bytes, ckv_stream stream);

/* Semantic Retrieval Score accumulation (Sec. 3.2, Eq. 5), the offline step that picks the
 * heads: srs[h] += sum over decode steps t whose generated token is in the answer span A of
 * sum_{j in A} a^h_{t,j}, for the layer's selected heads h (an all-ones head mask scores every
 * head).  Per sequence s of the batch (one profiling prompt each):
 *   k      [T, H_kv, d]: the context followed by the w generated tokens' keys; decode step t
 *          (t < w = cfg->window) attends to keys 0..L_s-w+t (itself included);
 *   q_dec  [S, w, H_q, d]: the decode steps' queries, laid out like q_win;
 *   lse    the decode rows' lse (natural log), layout as in ckv_score_window_lse;
 *   in_answer  device uint8 [S*w]: nonzero where step t's generated token is in A;
 *   span   device int32 [S][2]: A = positions [a0, a1) of the sequence (a span outside
 *          [0, L_s) is reported in the status word, kind 3, and skipped);
 *   srs    device fp32 [H_q], accumulated (+=) so that calls over prompts and layers add up.
 * The workspace is ckv_workspace_size's. */
CKV_API ckv_status ckv_semantic_retrieval_scores(const ckv_config* cfg, int32_t layer,
                                                 const ckv_batch* batch, const void* q_dec,
                                                 const void* k, int64_t tok_stride,
                                                 int64_t head_stride, const float* lse,
                                                 int64_t lse_head_stride, const uint8_t* in_answer,
                                                 const int32_t* span, float* srs, void* workspace,
                                                 size_t workspace_bytes, ckv_stream stream);

/* Layer budgets (App. B, the paper's error-aware layer-adaptive allocation).  Host only; no
 * GPU is needed.
 *
 * ckv_layer_error_scores: Eq. 11-13.  errors [num_datasets][num_layers] (host, row-major) are
 * the per-layer compression errors e_d^(l) of Eq. 10 (finite, >= 0; each dataset's row must
 * not sum to 0).  Each row is divided by its sum (Eq. 11), the rows are averaged (Eq. 12) and
 * the average is divided by its sum (Eq. 13) into scores[num_layers] (host, caller-owned).
 *
 * ckv_allocate_budgets: Algorithm 1.  From scores[num_layers] (finite, >= 0, normally the
 * output above) and the total budget B_total, every layer starts at min_budget (m), the rest
 * B_total - m * num_layers is handed out as round(score * rest) (ties to even) clipped to
 * [m, max_budget], and the difference left by rounding and clipping is settled one token at
 * a time: added to the highest-scoring layer still below M, or taken from the lowest-scoring
 * layer still above m (lowest layer index among equal scores).  The paper uses m = 32 and
 * M = 3 * B_total / num_layers.  The budgets sum to B_total whenever
 * m * num_layers <= B_total <= M * num_layers; otherwise every layer ends at m (or M).
 * Writes budgets[num_layers] (host, caller-owned), usable as ckv_config.budgets. */
CKV_API ckv_status ckv_layer_error_scores(const double* errors, int32_t num_datasets,
                                          int32_t num_layers, double* scores);
CKV_API ckv_status ckv_allocate_budgets(const double* scores, int32_t num_layers,
                                        int64_t total_budget, int32_t min_budget,
                                        int32_t max_budget, int32_t* budgets);

/* Limit, for the calls enqueued after this one, of every bounded wait in which a kernel
 * waits on another of its roles or on another CTA: 0 restores the default (about 2 s).  When
 * a wait runs out the kernel sets CKV_DEV status 2 (a wait gave up) in the workspace status
 * word, lets its own copies and MMAs finish, frees its tensor memory and returns; the results
 * of that call are then undefined, the CUDA context stays usable.  Process-wide; meant for
 * failure detection (and its tests), not for normal use. */
CKV_API ckv_status ckv_set_wait_limit_us(uint32_t microseconds);

/* Synchronises `stream`, then returns the workspace's device status: *code = 0 if no kernel
 * recorded an error since the last reset, else the first error (1 = cu_seqlens_dev disagrees
 * with the host copy, 2 = a wait timed out, 3 = an index out of range, 4 = a window row's
 * largest logit beyond +-680, which the two-pass kernel's fp64 row sums cannot hold); *detail
 * says where.
 * With reset != 0 the status word is cleared afterwards. */
CKV_API ckv_status ckv_read_device_status(void* workspace, ckv_stream stream, int32_t reset,
                                  int32_t* code, int32_t* detail);

/* ckv_score_window for callers that cannot allocate device memory (no counterpart in the
 * paper).  Some callers have no allocator to hand: code running inside a host-side engine
 * whose memory pool is owned elsewhere, or code that must not grow the process's device
 * footprint after start-up.  This variant takes no workspace.  Its scratch (the softmax
 * exchange of the scoring kernel -- per-item partials of the TMEM-resident kernel, or per-unit
 * sums of the two-pass kernel -- arrival counters and a status word) is a fixed, file-scope
 * device array of CKV_STATIC_SCRATCH_BYTES that every GPU loading the library holds until the
 * process exits.
 *   - Same arguments, results and layouts as ckv_score_window, minus the workspace.
 *   - The first call on a device looks up the array's device address (once per device, with
 *     that device current); make that first call before any stream capture.
 *   - Calls whose work needs more scratch than the array holds return CKV_ERR_UNSUPPORTED
 *     before enqueuing anything: on the resident kernel more than CKV_STATIC_SCRATCH_ITEMS
 *     work items over the call; on the two-pass kernel more than CKV_STATIC_SCRATCH_UNITS
 *     (head batch, sequence) units in one launch, which takes up to 256 sequences.
 *     ckv_score_window has no such limit.
 *   - Every call shares the one array: calls that may overlap on the GPU (other streams,
 *     other host threads) race and must be serialised by the caller.
 *   - Each call clears the status word first.  If status_out (device, 2 x int32) is not NULL,
 *     the call's device status (code, detail as in ckv_read_device_status) is copied there at
 *     the end of the call, in stream order.
 *   - Allocates nothing: no cudaMalloc, cudaFree or allocating library call. */
#define CKV_STATIC_SCRATCH_ITEMS 1024
#define CKV_STATIC_SCRATCH_UNITS 1024
#define CKV_STATIC_SCRATCH_BYTES (256 + CKV_STATIC_SCRATCH_ITEMS * 64 * 8 + 8192)
CKV_API ckv_status ckv_score_window_static(const ckv_config* cfg, int32_t layer,
                                           const ckv_batch* batch, const void* q_win,
                                           const void* k, int64_t tok_stride,
                                           int64_t head_stride, float* scores,
                                           int32_t* status_out, ckv_stream stream);

#ifdef __cplusplus
}
#endif

#endif /* CKV_H */
