// Host-side interface between the C ABI layer (ckv_api.cu) and the kernel launchers.
#pragma once

#include <cuda.h>
#include <cuda_runtime.h>
#include <stddef.h>
#include <stdint.h>

#include <vector>

#include <nvtx3/nvToolsExt.h>

namespace ckv {

// A host-side NVTX range around one kernel launch, named for the kernel, so that a profiler or
// timeline tool that attaches sees which library call each launch came from (ranges opened
// while a CUDA graph is captured mark the capture).  With no tool attached, the push and the pop
// go through NVTX's empty function table.
struct NvtxRange {
    explicit NvtxRange(const char* name) { nvtxRangePushA(name); }
    ~NvtxRange() { nvtxRangePop(); }
    NvtxRange(const NvtxRange&) = delete;
    NvtxRange& operator=(const NvtxRange&) = delete;
};

// A scoring work item: `ntiles` key tiles (128 keys each) of one unit, from tile `tile0`.
struct ScoreItem {
    uint16_t unit;     // index into the launch's unit table
    uint16_t ntiles;   // 0 = no work (round padding)
    uint32_t tile0;
};
// A scoring unit: one sequence x one batch of selected heads of a KV group.  Its items are
// contiguous in the item table and all belong to the same round.
struct ScoreUnit {
    int32_t seq_start;
    int32_t len;
    uint16_t seq;
    uint16_t batch;
    uint16_t first_item;  // relative to the launch
    uint16_t nitems;
};
constexpr int kMaxScoreItems = 2048;  // per launch (kernel-parameter table)
constexpr int kMaxScoreUnits = 384;

// A contiguous run of rounds that is launched together.
struct ScoreSlice {
    int item0, n_rounds, unit0, n_units;
};

struct ScoreLaunch {
    CUtensorMap tmap_k;
    CUtensorMap tmap_q;    // the window queries, boxes of w_pad rows x 64 dims
    const void* q_win;
    const int32_t* cu_seqlens_dev;
    void* partials;        // float2 [items per launch, n_cols]
    int* counters;         // [units per launch]
    float* scores;         // [n_sel, T]
    int* status;
    int S, T, Hq, w;
    int w_pad, n_cols;     // rows per head in the MMA (8/16/32/64), MMA N (32/64)
    int nb;                // head batches
    int grid;              // CTAs (= items per round)
    bool resident;         // score_resident.cu (logits kept in TMEM) instead of score_kernel.cu
    const float* lse;      // given window-row lse [Hq][lse_head_stride] (score_lse.cu), or null
    int64_t lse_head_stride;
    uint32_t cu_hash;      // seqlens_hash of the host copy of cu_seqlens
    float softmax_scale;
    int n_sel;
    const int* batch_group;
    const int* batch_first;
    const int* batch_nheads;
    const int* sel_heads;
    std::vector<ScoreItem> items;   // rounds x grid, units' items contiguous
    std::vector<ScoreUnit> units;   // first_item relative to the unit's slice
    std::vector<ScoreSlice> slices;
};
cudaError_t launch_score(const ScoreLaunch& L, cudaStream_t stream);

// Multi-layer scoring (score_layers.cu): both passes, K re-read from L2 in pass 2, every unit
// of every layer of the launch in one persistent cooperative kernel.  A unit is (head batch,
// sequence); its key tiles are split into m items of balanced length (m at most the launch's
// CTAs), and the CTAs take the items, unit after unit, from a global counter.
constexpr int kMaxLaunchLayers = 32;
constexpr int kMaxLaunchBatches = 256;   // head batches over the launch's layers
constexpr int kMaxLaunchSel = 512;       // head slots over the launch's layers
constexpr int kMaxLaunchSeqs = 256;
constexpr int kMaxLaunchUnits = 1536;
struct LaunchUnit {
    int16_t lb;      // flat head batch
    int16_t seq;     // sequence within the launch
    int32_t item0;   // first item; the unit's m items are item0 .. next unit's item0 - 1
};
struct LayersLayer {
    CUtensorMap tmap_k;
    CUtensorMap tmap_q;
    float* scores;       // [n_sel of the layer, T]
    const float* lse;    // the window rows' lse, [H_q][lse_stride] (given_lse launches)
    long long lse_stride;
};
struct LayersLaunch {
    std::vector<LayersLayer> layers;
    // flat over the layers' head batches, in layer order
    std::vector<int16_t> batch_layer, batch_group, batch_first, batch_nheads, batch_sel;
    std::vector<int16_t> sel_heads;  // query head of each head slot, batch after batch
    std::vector<int32_t> seq_start, seq_len;   // [S] of the launch's sequences seq0 ...
    std::vector<LaunchUnit> units;             // unit after unit, then one entry closing the table
    int seq0, S_all;     // the launch's first sequence; sequences in the batch (for the hash)
    const int32_t* cu_seqlens_dev;
    double* sums;        // [units][n_cols]
    int* counters;       // [units + 1]: arrivals per unit, then the item counter
    int* status;
    int T, w, w_pad, n_cols, grid;
    uint32_t cu_hash;
    float softmax_scale;
    bool given_lse;      // single pass with each layer's lse given (score_lse.cu)
};
cudaError_t launch_score_layers(const LayersLaunch& L, cudaStream_t stream);
long long wait_limit_cycles();  // the current limit of a bounded wait, in SM clock cycles

struct SelectLaunch {
    const float* scores;        // [n_sel, T]
    float* pooled;              // [H_kv, T]
    int32_t* idx;               // [H_kv, T_keep]
    int32_t* cu_keep_dev;       // [S+1]
    const int32_t* cu_seqlens_dev;
    int* status;
    int S, T, Hkv, w, budget, T_keep;
    int pool_kernel, pool_type, head_order;
    int skip_le;                // pooled is produced only for sequences with L > skip_le
    int from_scores;            // select: pool the scores on the fly (else read pooled)
    int write_pooled;           // with from_scores: also store the pooled scores (zeros
                                //   at window positions and unselected sequences)
    uint32_t cu_hash;
    const int* group_first;     // [n_vec+1] first score row of each selection's heads
    int n_vec;                  // selections per sequence: H_kv (per KV head) or 1 (per layer)
    int* hist;                  // [S*H_kv][select_hist_ints()] workspace, zero between calls
    int* arrivals;              // [S*H_kv] workspace, zero between calls
    int* chunk_start;           // [S*H_kv][max_chunks][select_hist_ints()] workspace
    void* buckets;              // [S*H_kv][max_chunks][select_chunk_positions()] 8-byte pairs
    int* info;                  // [S*H_kv][4] workspace
    int* chunk_off;             // [S*H_kv][max_chunks] workspace
    int max_chunks;             // select_chunks(longest sequence)
    int min_len, max_len;       // shortest and longest sequence (host lengths)
    const void* k;              // optional fused gather (nullptr: none)
    const void* v;
    int64_t tok_stride, head_stride;
    void* k_out;
    void* v_out;
    // The multi-layer selection: the scores viewed as 16-float lines (score_map_lines), with
    // 64 bytes of readable padding after the last row; nullptr: no such view.
    const CUtensorMap* score_map;
};
// Lines of 16 floats of a [n_sel, T] score buffer as the multi-layer selection's tensor map
// views it: every element, the last line's tail running into the padding after the buffer.
inline long long score_map_lines(int n_sel, int T) { return (static_cast<long long>(n_sel) * T + 15) / 16; }
constexpr int kScoreMapBoxLines = 176;  // lines per TMA box of the score map
int select_chunks(int max_len);
size_t select_hist_ints();
int select_chunk_positions();
int select_unit_len();  // units up to this length take the one-block path
cudaError_t launch_pool(const SelectLaunch& L, cudaStream_t stream);
cudaError_t launch_select(const SelectLaunch& L, cudaStream_t stream);
// The selections of several layers (one SelectLaunch each, pooling from their scores) in one
// launch per 32 layers: keys[i] is a [H_kv, select_key_stride(T, S)] scratch of 8-byte slots
// of layer i (each sequence's segment 32-byte aligned), next_unit a work counter (cleared by the
// call).
int select_key_stride(int T, int S);
cudaError_t launch_select_layers(const SelectLaunch* Ls, uint32_t* const* keys, int n_layers,
                                 int* next_unit, int grid, cudaStream_t stream);

struct GatherLaunch {
    const void* k;
    const void* v;
    int64_t tok_stride, head_stride;
    const int32_t* idx;
    const int32_t* cu_keep_dev;
    const int32_t* cu_seqlens_dev;
    void* k_out;
    void* v_out;
    int* status;
    int S, T, Hkv, T_keep;
    uint32_t cu_hash;
};
cudaError_t launch_gather(const GatherLaunch& L, cudaStream_t stream);

// Semantic Retrieval Score support (Eq. 5, srs_kernels.cu).
struct SrsLaunch {
    const float* lse;         // [Hq][lse_stride] the decode rows' lse
    int64_t lse_stride;
    const uint8_t* in_answer; // [S*w] the step's generated token is in the answer span
    float* lse_masked;        // [Hq][S*w] out: lse, or +inf where in_answer is 0
    const float* scores;      // [n_sel, T]
    const int32_t* span;      // [S][2] answer span [a0, a1), sequence-local
    const int32_t* cu_seqlens_dev;
    const int* sel_heads;     // host [n_sel]: query head of each score row
    float* srs;               // [Hq] accumulated
    int* status;
    int S, T, Hq, w, n_sel;
};
cudaError_t launch_srs_mask(const SrsLaunch& L, cudaStream_t stream);
cudaError_t launch_srs_span(const SrsLaunch& L, cudaStream_t stream);

int device_sm_count();

}  // namespace ckv
