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
    const float* scores;   // [n_sel, T]: pooled on the fly when from_scores != 0
    float* pooled;         // [H_kv, T]: read when from_scores == 0, else written if write_pooled
    int32_t* idx;
    int32_t* cu_keep;
    const int32_t* cu_seqlens;
    int* status;
    int S, T, Hkv, w, budget, T_keep;
    int pool_kernel, pool_type, head_order, from_scores, write_pooled;
    uint32_t cu_hash;
    int16_t group_first[kMaxQHeads + 1];
};

constexpr int kSelThreads = 1024;
constexpr int kSelWarps = kSelThreads / 32;
constexpr int kPoolTile = 8192;                         // candidate positions pooled per round
constexpr int kMaxHalo = kMaxPoolKernel / 2;
constexpr int kResidentKeys = 40960;                    // candidates kept in shared memory
constexpr int kSelSmemBytes = (kResidentKeys + kPoolTile + 2 * kMaxHalo) * 4;
static_assert(kPoolTile + 2 * kMaxHalo >= kSelWarps * 256, "per-warp histograms fit in the stage buffer");

// Order-preserving key of a non-negative float (-0 maps to +0).
__device__ __forceinline__ uint32_t rank_key(float f) {
    const uint32_t u = __float_as_uint(f);
    return u == 0x80000000u ? 0u : u;
}

// Block-wide exclusive prefix sum of v in thread order; *total gets the block's sum.
__device__ __forceinline__ int block_excl_scan(int v, int* scratch, int* total) {
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    int incl = v;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        const int y = __shfl_up_sync(0xffffffffu, incl, o);
        if (lane >= o) incl += y;
    }
    if (lane == 31) scratch[warp] = incl;
    __syncthreads();
    if (warp == 0) {
        const int x = lane < kSelWarps ? scratch[lane] : 0;
        int wincl = x;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const int y = __shfl_up_sync(0xffffffffu, wincl, o);
            if (lane >= o) wincl += y;
        }
        if (lane < kSelWarps) scratch[lane] = wincl - x;
        if (lane == 31) scratch[32] = wincl;
    }
    __syncthreads();
    const int r = scratch[warp] + incl - v;
    *total = scratch[32];
    __syncthreads();
    return r;
}

// One block per (sequence, KV head):
//   1. pooling of the selected heads' window scores along the candidate positions (max or avg,
//      zero padding outside [0, P)), in either head order, staged through shared memory;
//   2. radix select of the k-th largest pooled score (8-bit digits, most significant first)
//      over shared-memory keys;
//   3. a stable, position-ordered compaction: every candidate above the threshold and the
//      lowest-positioned ties, then the window positions.
__global__ void __launch_bounds__(kSelThreads, 1) pool_select_kernel(const __grid_constant__ SelectParams p) {
    extern __shared__ uint32_t sel_smem[];
    uint32_t* keys = sel_smem;                                               // [kResidentKeys]
    float* stage = reinterpret_cast<float*>(sel_smem + kResidentKeys);       // [kPoolTile + 2*halo]
    __shared__ int hist[256];
    __shared__ int scratch[33];
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
    if (L < 0 || t0 < 0 || keep_off < 0 || keep_off + n_keep > p.T_keep || t0 + L > p.T) {
        if (tid == 0) record_error(p.status, kDevBadSeqlens, 200 + s);
        return;
    }
    if (g == 0 && tid == 0) {
        p.cu_keep[s + 1] = keep_off + n_keep;
        if (s == 0) p.cu_keep[0] = 0;
    }
    int32_t* out = p.idx + static_cast<size_t>(g) * p.T_keep + keep_off;
    float* pooled = p.pooled ? p.pooled + static_cast<size_t>(g) * p.T + t0 : nullptr;
    if (L <= p.budget) {
        for (int i = tid; i < L; i += kSelThreads) {
            out[i] = i;
            if (p.from_scores && p.write_pooled) pooled[i] = 0.f;
        }
        return;
    }
    const int P = L - p.w, k = p.budget - p.w;
    const bool resident = P <= kResidentKeys;

    // ---------------------------------------------------------------- 1. pooling
    if (p.from_scores) {
        const int half = p.pool_kernel >> 1;
        const bool is_max = p.pool_type == 0;
        const float kf = static_cast<float>(p.pool_kernel);
        const int r0 = p.group_first[g], r1 = p.group_first[g + 1];
        const float* base = p.scores + t0;
        for (int tile0 = 0; tile0 < P; tile0 += kPoolTile) {
            const int n = min(kPoolTile, P - tile0);
            constexpr int kPer = kPoolTile / kSelThreads;
            float acc[kPer];
#pragma unroll
            for (int i = 0; i < kPer; ++i) acc[i] = 0.f;
            const int passes = p.head_order == 0 ? r1 - r0 : 1;
            for (int ps = 0; ps < passes; ++ps) {
                // stage positions tile0-half .. tile0+n+half (zeros outside [0, P)); every load
                // of a thread is issued before its stores, so the round trips overlap
                constexpr int kStagePer = (kPoolTile + 2 * kMaxHalo + kSelThreads - 1) / kSelThreads;
                float xs[kStagePer];
#pragma unroll
                for (int i = 0; i < kStagePer; ++i) {
                    const int e = tid + i * kSelThreads;
                    const int u = tile0 - half + e;
                    float x = 0.f;
                    if (e < n + 2 * half && u >= 0 && u < P) {
                        if (p.head_order == 0) {
                            x = __ldg(base + static_cast<size_t>(r0 + ps) * p.T + u);
                        } else {
                            for (int r = r0; r < r1; ++r) x += __ldg(base + static_cast<size_t>(r) * p.T + u);
                        }
                    }
                    xs[i] = x;
                }
#pragma unroll
                for (int i = 0; i < kStagePer; ++i) {
                    const int e = tid + i * kSelThreads;
                    if (e < n + 2 * half) stage[e] = xs[i];
                }
                __syncthreads();
#pragma unroll
                for (int i = 0; i < kPer; ++i) {
                    const int jl = tid + i * kSelThreads;  // window is stage[jl .. jl + 2*half]
                    if (jl < n) {
                        float m = stage[jl];
                        if (is_max) {
                            for (int t = 1; t <= 2 * half; ++t) m = fmaxf(m, stage[jl + t]);
                            acc[i] += m;
                        } else {
                            for (int t = 1; t <= 2 * half; ++t) m += stage[jl + t];
                            acc[i] += m / kf;  // IEEE division, as in pool_kernel
                        }
                    }
                }
                __syncthreads();
            }
#pragma unroll
            for (int i = 0; i < kPer; ++i) {
                const int jl = tid + i * kSelThreads;
                if (jl < n) {
                    if (resident) keys[tile0 + jl] = rank_key(acc[i]);
                    if (p.write_pooled || !resident) pooled[tile0 + jl] = acc[i];
                }
            }
        }
        if (p.write_pooled)
            for (int j = P + tid; j < L; j += kSelThreads) pooled[j] = 0.f;
    } else if (resident) {
        for (int j = tid; j < P; j += kSelThreads) keys[j] = rank_key(__ldg(pooled + j));
    }
    __syncthreads();
    // keys are either resident in shared memory or re-read from the pooled scores in global
    // memory (written above, visible to the block after the barrier)
    auto key_at = [&](int j) -> uint32_t {
        return resident ? keys[j] : rank_key(pooled[j]);
    };

    if (k > 0) {
        // ------------------------------------------------------------ 2. radix select
        uint32_t prefix = 0, mask = 0;
        int remaining = k;
        for (int shift = 24; shift >= 0; shift -= 8) {
            // Per-warp histograms (aliasing the pooling stage buffer): lanes with the same digit
            // are grouped by __match_any_sync and their leader adds the group's count, so
            // clustered scores neither serialise on shared atomics nor race across warps.
            int* whist = reinterpret_cast<int*>(stage) + (tid >> 5) * 256;
            const int lane = tid & 31;
#pragma unroll
            for (int b = lane; b < 256; b += 32) whist[b] = 0;
            __syncwarp();
            for (int j0 = 0; j0 < P; j0 += kSelThreads) {
                const int j = j0 + tid;
                const uint32_t u = j < P ? key_at(j) : 0u;
                const bool in = j < P && (u & mask) == prefix;
                const uint32_t digit = in ? ((u >> shift) & 255u) : 256u;
                const unsigned peers = __match_any_sync(0xffffffffu, digit);
                if (in && lane == __ffs(peers) - 1) whist[digit] += __popc(peers);
                __syncwarp();
            }
            __syncthreads();
            if (tid < 256) {
                int h = 0;
                const int* wh = reinterpret_cast<const int*>(stage) + tid;
#pragma unroll 8
                for (int w = 0; w < kSelWarps; ++w) h += wh[w * 256];
                hist[tid] = h;
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
                const int strictly_above = above - local;
                if (strictly_above < remaining && above >= remaining) {
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
        const uint32_t thr = prefix;    // the k-th largest key
        const int need_eq = remaining;  // ties at the threshold that are kept

        // ------------------------------------------------------------ 3. compaction
        const int seg = (P + kSelThreads - 1) / kSelThreads;
        const int j0 = min(P, tid * seg), j1 = min(P, j0 + seg);
        int n_gt = 0, n_eq = 0;
        for (int j = j0; j < j1; ++j) {
            const uint32_t u = key_at(j);
            n_gt += u > thr;
            n_eq += u == thr;
        }
        int tot;
        const int eq_before = block_excl_scan(n_eq, scratch, &tot);
        const int eq_take = max(0, min(n_eq, need_eq - eq_before));
        const int out_before = block_excl_scan(n_gt + eq_take, scratch, &tot);
        if (tid == 0 && tot != k) record_error(p.status, kDevBadIndex, 300 + blockIdx.x);
        int o = out_before, eq_seen = 0;
        for (int j = j0; j < j1; ++j) {
            const uint32_t u = key_at(j);
            const bool take = u > thr || (u == thr && eq_seen++ < eq_take);
            if (take && o < k) out[o++] = j;
        }
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
    p.scores = L.scores;
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
    p.pool_kernel = L.pool_kernel;
    p.pool_type = L.pool_type;
    p.head_order = L.head_order;
    p.from_scores = L.from_scores;
    p.write_pooled = L.write_pooled;
    p.cu_hash = L.cu_hash;
    for (int g = 0; g <= L.Hkv; ++g) p.group_first[g] = static_cast<int16_t>(L.group_first[g]);
    static bool configured = false;
    if (!configured) {
        cudaError_t e = cudaFuncSetAttribute(pool_select_kernel,
                                             cudaFuncAttributeMaxDynamicSharedMemorySize, kSelSmemBytes);
        if (e != cudaSuccess) return e;
        configured = true;
    }
    pool_select_kernel<<<L.S * L.Hkv, kSelThreads, kSelSmemBytes, stream>>>(p);
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
