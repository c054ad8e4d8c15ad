// The launch parameters and the work items shared by the two multi-layer scoring kernels: the
// two-pass kernel (score_layers.cu) and the single-pass kernel that takes the window rows' lse
// from the caller (score_lse.cu).
#pragma once

#include "score_common.cuh"

namespace ckv {

struct alignas(128) LayersParams {
    CUtensorMap tmap_k[kMaxLaunchLayers];  // K of each layer: {128, H_kv, T}, box {64, 1, 128}
    CUtensorMap tmap_q[kMaxLaunchLayers];  // q_win of each layer: {128, H_q, S*w}, box {64, 1, W_PAD}
    float* scores[kMaxLaunchLayers];       // [n_sel of the layer, T]
    const float* lse[kMaxLaunchLayers];    // given lse of each layer's window rows, [H_q][lse_stride]
    long long lse_stride[kMaxLaunchLayers];
    const int32_t* cu_seqlens;             // device [S+1] (checked against cu_hash)
    double* sums;                          // [n_units][N]: per column, sum of 2^(x) over the unit
    int* counters;                         // [n_units] arrivals, then the item counter; zero at launch
    int* status;
    int S, T, w, n_units, n_items, n_layers;
    int seq0, S_all;                       // the launch's first sequence, sequences of the batch
    uint32_t cu_hash;
    float sl2;                             // softmax scale * log2(e)
    long long wait_cycles;
    int16_t batch_layer[kMaxLaunchBatches];   // layer (launch-local) of each flat head batch
    int16_t batch_group[kMaxLaunchBatches];   // KV head
    int16_t batch_first[kMaxLaunchBatches];   // score row (in its layer) of the batch's first head
    int16_t batch_nheads[kMaxLaunchBatches];
    int16_t batch_sel[kMaxLaunchBatches];     // index into sel_heads of the batch's first head
    int16_t sel_heads[kMaxLaunchSel];         // query head of each head slot
    int32_t seq_start[kMaxLaunchSeqs];        // of the launch's sequences seq0, seq0 + 1, ...
    int32_t seq_len[kMaxLaunchSeqs];
    LaunchUnit units[kMaxLaunchUnits + 1];    // units[n_units].item0 = n_items
};
static_assert(sizeof(LayersParams) <= 32000, "kernel parameters");

struct Item {
    int layer, batch, seq, unit, tile0, ntiles, start, len, nitems;
};

// Item i of the launch: the unit whose items hold i, and the (i - item0)-th of its m balanced
// pieces of key tiles.
__device__ __forceinline__ Item get_item(const LayersParams& p, int i) {
    Item it;
    int lo = 0, hi = p.n_units - 1;  // the last unit whose first item is at or before i
    while (lo < hi) {
        const int mid = (lo + hi + 1) >> 1;
        if (p.units[mid].item0 <= i) lo = mid;
        else hi = mid - 1;
    }
    const LaunchUnit U = p.units[lo];
    const int m = p.units[lo + 1].item0 - U.item0;
    const int k = i - U.item0;
    it.unit = lo;
    it.batch = U.lb;
    it.layer = p.batch_layer[U.lb];
    it.seq = U.seq;
    it.start = p.seq_start[U.seq];
    it.len = p.seq_len[U.seq];
    it.nitems = m;
    const int tiles = (it.len + kTileKeys - 1) / kTileKeys;
    it.tile0 = k * tiles / m;
    it.ntiles = (k + 1) * tiles / m - it.tile0;
    return it;
}

// The index of the CTA's it-th item (-1 once its stream has ended), after the producer posted
// it into a ring of RING entries; false if the wait gave up.
template <int RING>
__device__ __forceinline__ bool wait_item(uint64_t* item_full, const int* items, int it, int* gi,
                                          volatile int* abort, long long lim) {
    const int k = it % RING;
    if (!mbar_wait(&item_full[k], (it / RING) & 1, abort, lim)) return false;
    *gi = items[k];
    return true;
}

// The single-pass multi-layer kernel (score_lse.cu): launch of one (N, W_PAD) instance.
cudaError_t dispatch_lse_layers(const LayersParams& p, int n_cols, int w_pad, int grid, cudaStream_t st);

}  // namespace ckv
