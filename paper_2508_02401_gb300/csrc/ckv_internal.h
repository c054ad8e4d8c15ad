// Host-side interface between the C ABI layer (ckv_api.cu) and the kernel launchers.
#pragma once

#include <cuda.h>
#include <cuda_runtime.h>
#include <stddef.h>
#include <stdint.h>

namespace ckv {

// One scoring launch pair (pass 1 -> partials, pass 2 -> scores).
struct ScoreLaunch {
    CUtensorMap tmap_k;
    const void* q_win;
    const int32_t* cu_seqlens_dev;
    void* partials;        // float2 [n_items, n_cols]
    float* scores;         // [n_sel, T]
    int* status;
    int S, T, Hq, w;
    int w_pad, n_cols;     // rows per head in the MMA (8/16/32/64), MMA N (32/64)
    int nb;                // head batches
    int n_items, chunk_tiles, grid;
    int skip_le;           // sequences with L <= skip_le are skipped (-1: none)
    uint32_t cu_hash;      // seqlens_hash of the host copy of cu_seqlens
    float softmax_scale;
    int n_sel;
    const int* batch_group;
    const int* batch_first;
    const int* batch_nheads;
    const int* sel_heads;
};
cudaError_t launch_score(const ScoreLaunch& L, cudaStream_t stream);

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
    int write_pooled;           // select with from_scores: also store the pooled scores
    uint32_t cu_hash;
    const int* group_first;     // [H_kv+1] first score row of each group
};
cudaError_t launch_pool(const SelectLaunch& L, cudaStream_t stream);
cudaError_t launch_select(const SelectLaunch& L, cudaStream_t stream);

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

int device_sm_count();

}  // namespace ckv
