// Pooling, top-N selection and the K/V gather (arxiv 2508.02401, Sec. 3.3 and Fig. 3): the
// window-summed scores are smoothed along the token axis, the selected heads' vectors of a KV
// group are combined, the N best-scoring positions are kept and their K/V rows are copied
// into the compacted cache.
#include "ckv_device.cuh"
#include "ckv_internal.h"

namespace ckv {

namespace {

struct PoolParams {
    const float* scores;
    float* pooled;
    const int32_t* cu_seqlens;
    int S, T, w, pool_kernel, pool_type, head_order, skip_le;
    int16_t group_first[kMaxQHeads + 1];
};

// Sequence containing token t: the last s with cu[s] <= t (cu non-decreasing).
__device__ __forceinline__ int seq_of(const int32_t* cu, int S, int t) {
    int lo = 0, hi = S - 1;
    while (lo < hi) {
        const int mid = (lo + hi + 1) >> 1;
        if (__ldg(cu + mid) <= t) lo = mid;
        else hi = mid - 1;
    }
    return lo;
}

// One thread per (token, KV head).  Pools over [j - k/2, j + k/2] clipped to the candidate
// range [0, P): max ignores the clipped cells, avg divides by the full kernel size.
__global__ void __launch_bounds__(256) pool_kernel(const __grid_constant__ PoolParams p) {
    const int t = blockIdx.x * blockDim.x + threadIdx.x;
    const int g = blockIdx.y;
    if (t >= p.T) return;
    const int s = seq_of(p.cu_seqlens, p.S, t);
    const int t0 = __ldg(p.cu_seqlens + s);
    const int L = __ldg(p.cu_seqlens + s + 1) - t0;
    const int P = L - p.w;
    const int j = t - t0;
    float out = 0.f;
    if (L > p.skip_le && j < P) {
        const int half = p.pool_kernel >> 1;
        const int lo = max(0, j - half), hi = min(P - 1, j + half);
        const int r0 = p.group_first[g], r1 = p.group_first[g + 1];
        const bool is_max = p.pool_type == 0;
        if (p.head_order == 0) {  // pool each head, then sum
            for (int r = r0; r < r1; ++r) {
                const float* a = p.scores + static_cast<size_t>(r) * p.T + t0;
                float acc = is_max ? __ldg(a + lo) : 0.f;
                for (int u = is_max ? lo + 1 : lo; u <= hi; ++u)
                    acc = is_max ? fmaxf(acc, __ldg(a + u)) : acc + __ldg(a + u);
                out += is_max ? acc : acc / static_cast<float>(p.pool_kernel);
            }
        } else {  // sum heads, then pool
            float acc = 0.f;
            for (int u = lo; u <= hi; ++u) {
                float x = 0.f;
                for (int r = r0; r < r1; ++r) x += __ldg(p.scores + static_cast<size_t>(r) * p.T + t0 + u);
                acc = (is_max && u > lo) ? fmaxf(acc, x) : (is_max ? x : acc + x);
            }
            out = is_max ? acc : acc / static_cast<float>(p.pool_kernel);
        }
    }
    p.pooled[static_cast<size_t>(g) * p.T + t] = out;
}

struct SelectParams {
    const float* pooled;
    int32_t* idx;
    int32_t* cu_keep;
    const int32_t* cu_seqlens;
    int* status;
    int S, T, Hkv, w, budget, T_keep;
    uint32_t cu_hash;
};

constexpr int kSelThreads = 1024;

// Order-preserving key of a non-negative float (-0 maps to +0).
__device__ __forceinline__ uint32_t rank_key(float f) {
    const uint32_t u = __float_as_uint(f);
    return u == 0x80000000u ? 0u : u;
}

// Block-wide exclusive count of `flag` in thread order; returns the rank, *total the sum.
__device__ __forceinline__ int block_rank(bool flag, int* warp_tot, int* total) {
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const unsigned bal = __ballot_sync(0xffffffffu, flag);
    const int in_warp = __popc(bal & ((1u << lane) - 1u));
    if (lane == 0) warp_tot[warp] = __popc(bal);
    __syncthreads();
    if (warp == 0) {
        const int x = warp_tot[lane];
        int incl = x;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const int y = __shfl_up_sync(0xffffffffu, incl, o);
            if (lane >= o) incl += y;
        }
        warp_tot[lane] = incl - x;                    // exclusive warp offsets
        if (lane == 31) warp_tot[32] = incl;          // block total
    }
    __syncthreads();
    const int r = warp_tot[warp] + in_warp;
    *total = warp_tot[32];
    __syncthreads();
    return r;
}

// One block per (sequence, KV head): radix select of the k-th largest pooled score (8-bit
// digits, most significant first), then a stable, position-ordered compaction that takes
// every score above the threshold and the lowest-positioned ties, then the window.
__global__ void __launch_bounds__(kSelThreads) select_kernel(const __grid_constant__ SelectParams p) {
    __shared__ int hist[256];
    __shared__ int warp_tot[33];
    __shared__ int s_digit, s_above;

    const int s = blockIdx.x / p.Hkv, g = blockIdx.x % p.Hkv;
    const int tid = threadIdx.x;
    if (blockIdx.x == 0 && tid == 0 && seqlens_hash(p.cu_seqlens, p.S) != p.cu_hash)
        record_error(p.status, kDevBadSeqlens, 200);
    const int t0 = p.cu_seqlens[s];
    const int L = p.cu_seqlens[s + 1] - t0;
    int keep_off = 0;
    for (int u = 0; u < s; ++u) keep_off += min(p.budget, p.cu_seqlens[u + 1] - p.cu_seqlens[u]);
    const int n_keep = min(p.budget, L);
    if (L < 0 || keep_off + n_keep > p.T_keep || t0 + L > p.T) {
        if (tid == 0) record_error(p.status, kDevBadSeqlens, 200 + s);
        return;
    }
    if (g == 0 && tid == 0) {
        p.cu_keep[s + 1] = keep_off + n_keep;
        if (s == 0) p.cu_keep[0] = 0;
    }
    int32_t* out = p.idx + static_cast<size_t>(g) * p.T_keep + keep_off;
    if (L <= p.budget) {
        for (int i = tid; i < L; i += kSelThreads) out[i] = i;
        return;
    }
    const int P = L - p.w, k = p.budget - p.w;
    const float* c = p.pooled + static_cast<size_t>(g) * p.T + t0;

    if (k > 0) {
        uint32_t prefix = 0, mask = 0;
        int remaining = k;
        for (int shift = 24; shift >= 0; shift -= 8) {
            if (tid < 256) hist[tid] = 0;
            __syncthreads();
            for (int j = tid; j < P; j += kSelThreads) {
                const uint32_t u = rank_key(__ldg(c + j));
                if ((u & mask) == prefix) atomicAdd(&hist[(u >> shift) & 255u], 1);
            }
            __syncthreads();
            if (tid < 32) {
                // lane l owns bins 8l .. 8l+7; find the digit where the count from the top
                // first reaches `remaining`
                int local = 0;
#pragma unroll
                for (int b = 0; b < 8; ++b) local += hist[tid * 8 + b];
                int above = local;  // inclusive suffix sum over lanes >= tid
#pragma unroll
                for (int o = 1; o < 32; o <<= 1) {
                    const int y = __shfl_down_sync(0xffffffffu, above, o);
                    if (tid + o < 32) above += y;
                }
                const int strictly_above = above - local;  // bins of higher lanes
                const bool here = strictly_above < remaining && above >= remaining;
                if (here) {
                    int acc = strictly_above;
                    for (int b = 7; b >= 0; --b) {
                        const int h = hist[tid * 8 + b];
                        if (acc + h >= remaining) {
                            s_digit = tid * 8 + b;
                            s_above = acc;
                            break;
                        }
                        acc += h;
                    }
                }
            }
            __syncthreads();
            prefix |= static_cast<uint32_t>(s_digit) << shift;
            mask |= 255u << shift;
            remaining -= s_above;
            __syncthreads();
        }
        const uint32_t thr = prefix;  // the k-th largest key
        const int need_eq = remaining;  // ties at the threshold that are kept
        int written = 0, eq_seen = 0;
        for (int j0 = 0; j0 < P; j0 += kSelThreads) {
            const int j = j0 + tid;
            const uint32_t u = j < P ? rank_key(__ldg(c + j)) : 0u;
            const bool gt = j < P && u > thr;
            const bool eq = j < P && u == thr;
            int eq_tot;
            const int eq_rank = block_rank(eq, warp_tot, &eq_tot);
            const bool take = gt || (eq && eq_seen + eq_rank < need_eq);
            int take_tot;
            const int out_rank = block_rank(take, warp_tot, &take_tot);
            if (take && written + out_rank < k) out[written + out_rank] = j;
            written += take_tot;
            eq_seen += eq_tot;
        }
        if (tid == 0 && written != k) record_error(p.status, kDevBadIndex, 300 + blockIdx.x);
    }
    for (int i = tid; i < p.w; i += kSelThreads) out[k + i] = P + i;
}

struct GatherParams {
    const uint4* k;
    const uint4* v;
    int64_t tok_stride, head_stride;  // in 16-byte units
    const int32_t* idx;
    const int32_t* cu_keep;
    const int32_t* cu_seqlens;
    uint4* k_out;
    uint4* v_out;
    int* status;
    int S, T, Hkv, T_keep;
    uint32_t cu_hash;
};

// One warp per kept (token, KV head) row: lanes 0-15 copy the 256-byte K row, lanes 16-31
// the V row, 16 bytes each.
__global__ void __launch_bounds__(256) gather_kernel(const __grid_constant__ GatherParams p) {
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const long long row = static_cast<long long>(blockIdx.x) * 8 + warp;
    if (row == 0 && lane == 0 && seqlens_hash(p.cu_seqlens, p.S) != p.cu_hash)
        record_error(p.status, kDevBadSeqlens, 400);
    if (row >= static_cast<long long>(p.T_keep) * p.Hkv) return;
    const int i = static_cast<int>(row / p.Hkv), g = static_cast<int>(row % p.Hkv);
    const int s = seq_of(p.cu_keep, p.S, i);
    const int pos = __ldg(p.idx + static_cast<size_t>(g) * p.T_keep + i);
    const int t0 = __ldg(p.cu_seqlens + s);
    const int L = __ldg(p.cu_seqlens + s + 1) - t0;
    if (pos < 0 || pos >= L || t0 + L > p.T) {
        if (lane == 0) record_error(p.status, kDevBadIndex, 400 + s);
        return;
    }
    const int part = lane & 15;
    const uint4* src = (lane < 16 ? p.k : p.v) + (t0 + pos) * p.tok_stride + g * p.head_stride + part;
    uint4* dst = (lane < 16 ? p.k_out : p.v_out) + row * 16 + part;
    *dst = __ldg(src);
}

}  // namespace

cudaError_t launch_pool(const SelectLaunch& L, cudaStream_t stream) {
    PoolParams p;
    p.scores = L.scores;
    p.pooled = L.pooled;
    p.cu_seqlens = L.cu_seqlens_dev;
    p.S = L.S;
    p.T = L.T;
    p.w = L.w;
    p.pool_kernel = L.pool_kernel;
    p.pool_type = L.pool_type;
    p.head_order = L.head_order;
    p.skip_le = L.skip_le;
    for (int g = 0; g <= L.Hkv; ++g) p.group_first[g] = static_cast<int16_t>(L.group_first[g]);
    if (L.T == 0) return cudaSuccess;
    dim3 grid((L.T + 255) / 256, L.Hkv);
    pool_kernel<<<grid, 256, 0, stream>>>(p);
    return cudaGetLastError();
}

cudaError_t launch_select(const SelectLaunch& L, cudaStream_t stream) {
    SelectParams p;
    p.pooled = L.pooled;
    p.idx = L.idx;
    p.cu_keep = L.cu_keep_dev;
    p.cu_seqlens = L.cu_seqlens_dev;
    p.status = L.status;
    p.S = L.S;
    p.T = L.T;
    p.Hkv = L.Hkv;
    p.w = L.w;
    p.budget = L.budget;
    p.T_keep = L.T_keep;
    p.cu_hash = L.cu_hash;
    select_kernel<<<L.S * L.Hkv, kSelThreads, 0, stream>>>(p);
    return cudaGetLastError();
}

cudaError_t launch_gather(const GatherLaunch& L, cudaStream_t stream) {
    GatherParams p;
    p.k = reinterpret_cast<const uint4*>(L.k);
    p.v = reinterpret_cast<const uint4*>(L.v);
    p.tok_stride = L.tok_stride / 8;
    p.head_stride = L.head_stride / 8;
    p.idx = L.idx;
    p.cu_keep = L.cu_keep_dev;
    p.cu_seqlens = L.cu_seqlens_dev;
    p.k_out = reinterpret_cast<uint4*>(L.k_out);
    p.v_out = reinterpret_cast<uint4*>(L.v_out);
    p.status = L.status;
    p.S = L.S;
    p.T = L.T;
    p.Hkv = L.Hkv;
    p.T_keep = L.T_keep;
    p.cu_hash = L.cu_hash;
    const long long rows = static_cast<long long>(L.T_keep) * L.Hkv;
    if (rows == 0) return cudaSuccess;
    gather_kernel<<<static_cast<unsigned>((rows + 7) / 8), 256, 0, stream>>>(p);
    return cudaGetLastError();
}

}  // namespace ckv
