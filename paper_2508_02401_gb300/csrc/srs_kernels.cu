// Semantic Retrieval Score accumulation (arxiv 2508.02401, Sec. 3.2, Eq. 5):
//
//   SRS(h) += sum over decode steps t with y_t in A of  sum_{j in A} a^h_{t,j}
//
// computed with the window-scoring machinery: the decode steps' queries are the window rows
// over a key buffer that holds the context followed by the generated tokens, so step t sees
// keys 0..L-w+t (itself included), and the steps whose generated token is not in the answer
// span get lse = +inf, which makes their probabilities 0.  The score row of head h then holds
// sum_t [y_t in A] a^h_{t,j} for every key j, and SRS(h) is its sum over the span.
#include "ckv_device.cuh"
#include "ckv_internal.h"

#include <math.h>
#include <string.h>

#include <algorithm>

namespace ckv {
namespace {

constexpr int kMaxSrsHeads = 256;

__global__ void srs_mask_kernel(const float* __restrict__ lse, long long lse_stride,
                                const uint8_t* __restrict__ in_answer, float* __restrict__ out,
                                int Hq, int rows) {
    const int64_t n = static_cast<int64_t>(Hq) * rows;
    for (int64_t i = blockIdx.x * static_cast<int64_t>(blockDim.x) + threadIdx.x; i < n;
         i += static_cast<int64_t>(gridDim.x) * blockDim.x) {
        const int h = static_cast<int>(i / rows), r = static_cast<int>(i % rows);
        out[i] = in_answer[r] ? lse[h * lse_stride + r] : INFINITY;
    }
}

struct SpanParams {
    const float* scores;
    const int32_t* span;
    const int32_t* cu_seqlens;
    float* srs;
    int* status;
    int T, S;
    int16_t sel_heads[kMaxSrsHeads];
};

// Block (score row i, sequence s): the sum of the row over the sequence's answer span, added
// to srs[query head of row i].  A span outside [0, L) is reported (status) and skipped.
__global__ void __launch_bounds__(256) srs_span_kernel(const __grid_constant__ SpanParams p) {
    const int i = blockIdx.x, s = blockIdx.y;
    const int t0 = __ldg(p.cu_seqlens + s), L = __ldg(p.cu_seqlens + s + 1) - t0;
    const int a0 = __ldg(p.span + 2 * s), a1 = __ldg(p.span + 2 * s + 1);
    if (a0 < 0 || a1 < a0 || a1 > L) {
        if (threadIdx.x == 0) record_error(p.status, kDevBadIndex, 500 + s);
        return;
    }
    const float* row = p.scores + static_cast<size_t>(i) * p.T + t0;
    float acc = 0.f;
    for (int j = a0 + threadIdx.x; j < a1; j += blockDim.x) acc += row[j];
    acc = warp_sum(acc);
    __shared__ float part[8];
    if ((threadIdx.x & 31) == 0) part[threadIdx.x >> 5] = acc;
    __syncthreads();
    if (threadIdx.x == 0) {
        float tot = 0.f;
        for (int q = 0; q < 8; ++q) tot += part[q];
        atomicAdd(p.srs + p.sel_heads[i], tot);
    }
}

}  // namespace

cudaError_t launch_srs_mask(const SrsLaunch& L, cudaStream_t stream) {
    const int rows = L.S * L.w;
    const int64_t n = static_cast<int64_t>(L.Hq) * rows;
    if (n == 0) return cudaSuccess;
    const int blocks = static_cast<int>(std::min<int64_t>((n + 255) / 256, 4096));
    NvtxRange range("srs_mask_kernel");
    srs_mask_kernel<<<blocks, 256, 0, stream>>>(L.lse, L.lse_stride, L.in_answer, L.lse_masked, L.Hq, rows);
    return cudaGetLastError();
}

cudaError_t launch_srs_span(const SrsLaunch& L, cudaStream_t stream) {
    if (L.n_sel == 0 || L.S == 0) return cudaSuccess;
    if (L.n_sel > kMaxSrsHeads || L.S > 65535) return cudaErrorInvalidValue;
    SpanParams p;
    memset(&p, 0, sizeof p);
    p.scores = L.scores;
    p.span = L.span;
    p.cu_seqlens = L.cu_seqlens_dev;
    p.srs = L.srs;
    p.status = L.status;
    p.T = L.T;
    p.S = L.S;
    for (int i = 0; i < L.n_sel; ++i) p.sel_heads[i] = static_cast<int16_t>(L.sel_heads[i]);
    NvtxRange range("srs_span_kernel");
    srs_span_kernel<<<dim3(L.n_sel, L.S), 256, 0, stream>>>(p);
    return cudaGetLastError();
}

}  // namespace ckv
