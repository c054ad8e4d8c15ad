// Pooling, top-N selection and the K/V gather (arxiv 2508.02401, Sec. 3.3 and Fig. 3): the
// window-summed scores are smoothed along the token axis, the selected heads' vectors of a KV
// group are combined, the N best-scoring positions are kept and their K/V rows are copied
// into the compacted cache.
#include "ckv_device.cuh"
#include "ckv_internal.h"

#include <limits.h>
#include <string.h>

#include <mutex>

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

// ------------------------------------------------------------------------ selection
// Three kernels per call, each over (sequence, KV head) units:
//   pool_hist   grid (unit, chunk): pools one chunk of kChunk candidate positions and adds the
//               chunk's histogram of the top 11 bits of the order-preserving score keys to the
//               unit's histogram in the workspace;
//   threshold   one block per unit: the exact k-th largest key, the position up to which the
//               keys equal to it are kept (lowest positions first, as a stable sort by
//               descending score would keep them), and each chunk's output offset;
//   compact     grid (unit, chunk): writes the chunk's kept positions in position order and,
//               when asked, copies their K/V rows into the compacted cache; chunk 0 also
//               writes the window.
// The histogram is zero outside a call: threshold clears each unit's copy once it has read it.
constexpr int kChunk = 4096;                 // candidate positions per chunk
constexpr int kChunkShift = 12;
constexpr int kHistBins = 2048;              // digits of up to 11 bits
constexpr int kHistShift = 21;               // the first digit is bits 31..21 of a key
constexpr int kPHThreads = 512;              // pool_hist and compact
constexpr int kPHPer = kChunk / kPHThreads;  // positions per thread
constexpr int kPHWarps = kPHThreads / 32;
constexpr int kWarpSpan = kChunk / kPHWarps; // compact: contiguous positions per warp
constexpr int kMaxHalo = kMaxPoolKernel / 2;
constexpr int kStageFloats = kChunk + 2 * kMaxHalo;
constexpr int kThThreads = 1024;             // threshold
constexpr int kCandCap = 8192;               // threshold: candidates kept in shared memory
constexpr int kCompactSmem = kChunk * 4;     // compact: the chunk's kept positions
constexpr uint32_t kTaken = 0xFFFFFFFEu;     // candidate markers (the top bit excludes them
constexpr uint32_t kDropped = 0xFFFFFFFFu;   // from the tie-position select)
static_assert(kWarpSpan % 32 == 0 && (1 << kChunkShift) == kChunk, "chunk shape");

struct SelectParams {
    const float* scores;   // [n_sel, T]: pooled in pool_hist when from_scores != 0
    float* pooled;         // [H_kv, T]
    int32_t* idx;          // [H_kv, T_keep]
    int32_t* cu_keep;      // [S+1]
    const int32_t* cu_seqlens;
    int* status;
    int* hist;             // [units][kHistBins]
    int* info;             // [units][4]: threshold key, tie cutoff position
    int* chunk_off;        // [units][max_chunks]: output offset of each chunk's kept positions
    const uint4* k;        // gather source (nullptr: no gather); strides in 16-byte units
    const uint4* v;
    int64_t tok_stride, head_stride;
    uint4* k_out;
    uint4* v_out;
    int S, T, Hkv, w, budget, T_keep, max_chunks;
    int pool_kernel, pool_type, head_order, from_scores, write_pooled;
    uint32_t cu_hash;
    int16_t group_first[kMaxQHeads + 1];
};

// Order-preserving unsigned key of a float (-0 and +0 share one key).
__device__ __forceinline__ uint32_t rank_key(float f) {
    uint32_t u = __float_as_uint(f);
    if (u == 0x80000000u) u = 0u;
    return (u & 0x80000000u) ? ~u : (u | 0x80000000u);
}

struct UnitGeo {
    int s, g, t0, L, P, k, keep_off, n_keep;
};

// Geometry of unit (sequence s, KV head g), from the device cu_seqlens; false (and an error
// recorded) if they are unusable.  Every thread of the block calls it.
__device__ __forceinline__ bool unit_geo(const SelectParams& p, int unit, UnitGeo& u) {
    u.s = unit / p.Hkv;
    u.g = unit % p.Hkv;
    u.t0 = __ldg(p.cu_seqlens + u.s);
    u.L = __ldg(p.cu_seqlens + u.s + 1) - u.t0;
    int off = 0;  // kept tokens of the earlier sequences: lanes stride over them
    for (int x = threadIdx.x & 31; x < u.s; x += 32)
        off += min(p.budget, __ldg(p.cu_seqlens + x + 1) - __ldg(p.cu_seqlens + x));
    off = __reduce_add_sync(0xffffffffu, off);
    u.keep_off = off;
    u.n_keep = min(p.budget, u.L);
    u.P = u.L - p.w;
    u.k = p.budget - p.w;
    if (u.L < 0 || u.t0 < 0 || u.t0 + u.L > p.T || off < 0 || off + u.n_keep > p.T_keep) {
        if (threadIdx.x == 0) record_error(p.status, kDevBadSeqlens, 200 + u.s);
        return false;
    }
    return true;
}

// Block-wide exclusive prefix sum over NT threads in thread order; *total gets the sum.
template <int NT>
__device__ __forceinline__ int block_excl_scan(int v, int* scratch, int* total) {
    constexpr int NW = NT / 32;
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
        const int x = lane < NW ? scratch[lane] : 0;
        int wincl = x;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const int y = __shfl_up_sync(0xffffffffu, wincl, o);
            if (lane >= o) wincl += y;
        }
        if (lane < NW) scratch[lane] = wincl - x;
        if (lane == 31) scratch[32] = wincl;
    }
    __syncthreads();
    const int r = scratch[warp] + incl - v;
    *total = scratch[32];
    __syncthreads();
    return r;
}

// Copies the K and V rows of sequence-local positions list[0..m) to output rows
// out_row0 + 0..m-1 of KV head g: a warp per row (16 lanes for K, 16 for V), four rows in
// flight per warp.
__device__ __forceinline__ void copy_rows(const SelectParams& p, const UnitGeo& u, const int* list,
                                          int m, int out_row0) {
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31, nw = blockDim.x >> 5;
    const int part = lane & 15;
    const uint4* src0 = (lane < 16 ? p.k : p.v) + static_cast<int64_t>(u.t0) * p.tok_stride +
                        static_cast<int64_t>(u.g) * p.head_stride + part;
    uint4* dst0 = (lane < 16 ? p.k_out : p.v_out) + static_cast<int64_t>(u.g) * 16 + part;
    for (int e0 = warp; e0 < m; e0 += 4 * nw) {
        uint4 x[4];
#pragma unroll
        for (int q = 0; q < 4; ++q) {
            const int e = e0 + q * nw;
            if (e < m) x[q] = __ldg(src0 + static_cast<int64_t>(list[e]) * p.tok_stride);
        }
#pragma unroll
        for (int q = 0; q < 4; ++q) {
            const int e = e0 + q * nw;
            if (e < m) dst0[static_cast<int64_t>(out_row0 + e) * p.Hkv * 16] = x[q];
        }
    }
}

__global__ void __launch_bounds__(kPHThreads) pool_hist_kernel(const __grid_constant__ SelectParams p) {
    extern __shared__ float stage[];  // [kStageFloats]
    __shared__ int hist[kHistBins];
    const int unit = blockIdx.x, c = blockIdx.y, tid = threadIdx.x, lane = tid & 31;
    if (unit == 0 && c == 0 && tid == 0 && seqlens_hash(p.cu_seqlens, p.S) != p.cu_hash)
        record_error(p.status, kDevBadSeqlens, 200);
    UnitGeo u;
    if (!unit_geo(p, unit, u)) return;
    float* pooled = p.pooled + static_cast<size_t>(u.g) * p.T + u.t0;
    const int j0 = c * kChunk;
    const bool zeros = p.from_scores && p.write_pooled;
    if (u.L <= p.budget) {  // kept whole: nothing to select; its pooled scores read as 0
        if (zeros)
            for (int j = j0 + tid; j < min(u.L, j0 + kChunk); j += kPHThreads) pooled[j] = 0.f;
        return;
    }
    if (zeros)  // window positions are not candidates
        for (int j = max(j0, u.P) + tid; j < min(u.L, j0 + kChunk); j += kPHThreads) pooled[j] = 0.f;
    if (j0 >= u.P) return;
    const int n = min(kChunk, u.P - j0);
    float acc[kPHPer];
#pragma unroll
    for (int i = 0; i < kPHPer; ++i) acc[i] = 0.f;
    if (p.from_scores) {
        // Same arithmetic, in the same order, as pool_kernel: the zeros staged outside [0, P)
        // leave a max of non-negative scores and a sum unchanged.
        const int half = p.pool_kernel >> 1;
        const bool is_max = p.pool_type == 0;
        const float kf = static_cast<float>(p.pool_kernel);
        const int r0 = p.group_first[u.g], r1 = p.group_first[u.g + 1];
        const float* base = p.scores + u.t0;
        const int passes = p.head_order == 0 ? r1 - r0 : 1;
        for (int ps = 0; ps < passes; ++ps) {
            // stage positions j0-half .. j0+n+half-1; each thread issues all its loads first
            constexpr int kStagePer = (kStageFloats + kPHThreads - 1) / kPHThreads;
            float xs[kStagePer];
#pragma unroll
            for (int i = 0; i < kStagePer; ++i) {
                const int e = tid + i * kPHThreads;
                const int uu = j0 - half + e;
                float x = 0.f;
                if (e < n + 2 * half && uu >= 0 && uu < u.P) {
                    if (p.head_order == 0) {
                        x = __ldg(base + static_cast<size_t>(r0 + ps) * p.T + uu);
                    } else {
                        for (int r = r0; r < r1; ++r) x += __ldg(base + static_cast<size_t>(r) * p.T + uu);
                    }
                }
                xs[i] = x;
            }
#pragma unroll
            for (int i = 0; i < kStagePer; ++i) {
                const int e = tid + i * kPHThreads;
                if (e < n + 2 * half) stage[e] = xs[i];
            }
            __syncthreads();
#pragma unroll
            for (int i = 0; i < kPHPer; ++i) {
                const int jl = tid + i * kPHThreads;  // its window: stage[jl .. jl + 2*half]
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
        for (int i = 0; i < kPHPer; ++i) {
            const int jl = tid + i * kPHThreads;
            if (jl < n) pooled[j0 + jl] = acc[i];
        }
    } else {
#pragma unroll
        for (int i = 0; i < kPHPer; ++i) {
            const int jl = tid + i * kPHThreads;
            acc[i] = jl < n ? __ldg(pooled + j0 + jl) : 0.f;
        }
    }
    // the chunk's histogram of the first digit, then into the unit's histogram
    for (int b = tid; b < kHistBins; b += kPHThreads) hist[b] = 0;
    __syncthreads();
#pragma unroll
    for (int i = 0; i < kPHPer; ++i) {
        const int jl = tid + i * kPHThreads;
        const bool in = jl < n;
        const uint32_t bin = in ? (rank_key(acc[i]) >> kHistShift) : static_cast<uint32_t>(kHistBins);
        const unsigned peers = __match_any_sync(0xffffffffu, bin);
        if (in && lane == __ffs(peers) - 1) atomicAdd(&hist[bin], __popc(peers));
    }
    __syncthreads();
    int* gh = p.hist + static_cast<size_t>(unit) * kHistBins;
    for (int b = tid; b < kHistBins; b += kPHThreads) {
        const int h = hist[b];
        if (h) atomicAdd(gh + b, h);
    }
}

// The digit d of a kHistBins-bin histogram with count(bins above d) < r <= count(bins >= d)
// (r >= 1): *s_digit = d, *s_above = count(bins above d).  Thread 0 owns the highest bins.
__device__ __forceinline__ void find_digit(const int* hist, int r, int* scratch, int* s_digit,
                                           int* s_above) {
    constexpr int PER = kHistBins / kThThreads;
    if (threadIdx.x == 0) {
        *s_digit = 0;
        *s_above = 0;
    }
    const int base = (kThThreads - 1 - static_cast<int>(threadIdx.x)) * PER;
    int local = 0;
#pragma unroll
    for (int q = 0; q < PER; ++q) local += hist[base + q];
    int tot;
    const int above = block_excl_scan<kThThreads>(local, scratch, &tot);
    if (above < r && above + local >= r) {
        int acc = above;
        for (int q = PER - 1; q >= 0; --q) {
            const int h = hist[base + q];
            if (acc + h >= r) {
                *s_digit = base + q;
                *s_above = acc;
                break;
            }
            acc += h;
        }
    }
    __syncthreads();
}

struct SelectState {
    int hist[kHistBins];
    int scratch[33];
    int digit, above, n_cand, cut_chunk, cut_take, cut_pos;
};

// The r-th largest (r >= 1) of the values vals[0..n) whose bits under `mask` equal `prefix`,
// found digit by digit over the `bits` lower bits.  *r_eq gets how many of the copies of the
// result rank within the first r, *n_eq how many copies there are.
__device__ uint32_t smem_select(const uint32_t* vals, int n, uint32_t prefix, uint32_t mask, int bits,
                                int r, SelectState& st, int* r_eq, int* n_eq) {
    const int tid = threadIdx.x, lane = tid & 31;
    int last = 0;
    while (bits > 0) {
        const int d = bits > 11 ? 11 : bits;
        const int shift = bits - d;
        const uint32_t dmask = (1u << d) - 1u;
        for (int b = tid; b < kHistBins; b += kThThreads) st.hist[b] = 0;
        __syncthreads();
        for (int i0 = 0; i0 < n; i0 += kThThreads) {
            const int i = i0 + tid;
            const uint32_t x = i < n ? vals[i] : 0u;
            const bool in = i < n && (x & mask) == prefix;
            const uint32_t bin = in ? (x >> shift) & dmask : static_cast<uint32_t>(kHistBins);
            const unsigned peers = __match_any_sync(0xffffffffu, bin);
            if (in && lane == __ffs(peers) - 1) atomicAdd(&st.hist[bin], __popc(peers));
        }
        __syncthreads();
        find_digit(st.hist, r, st.scratch, &st.digit, &st.above);
        const int dg = st.digit;
        last = st.hist[dg];
        prefix |= static_cast<uint32_t>(dg) << shift;
        mask |= dmask << shift;
        r -= st.above;
        bits -= d;
        __syncthreads();  // everyone has read hist and digit before they are reused
    }
    *r_eq = r;
    *n_eq = last;
    return prefix;
}

__global__ void __launch_bounds__(kThThreads, 1) threshold_kernel(const __grid_constant__ SelectParams p) {
    extern __shared__ uint32_t th_smem[];  // cand_key[kCandCap] cand_pos[kCandCap] cnt eqc [max_chunks]
    __shared__ SelectState st;
    uint32_t* cand_key = th_smem;
    int* cand_pos = reinterpret_cast<int*>(th_smem + kCandCap);
    int* cnt = reinterpret_cast<int*>(th_smem + 2 * kCandCap);
    int* eqc = cnt + p.max_chunks;
    const int unit = blockIdx.x, tid = threadIdx.x, lane = tid & 31;
    // take the unit's first-digit histogram and leave zeros behind for the next call
    int* gh = p.hist + static_cast<size_t>(unit) * kHistBins;
    for (int b = tid; b < kHistBins; b += kThThreads) {
        st.hist[b] = __ldcg(gh + b);
        __stcg(gh + b, 0);
    }
    UnitGeo u;
    if (!unit_geo(p, unit, u)) return;
    if (u.L <= p.budget) return;
    const int P = u.P, k = u.k, nch = (P + kChunk - 1) / kChunk;
    int* info = p.info + unit * 4;
    int* coff = p.chunk_off + static_cast<size_t>(unit) * p.max_chunks;
    if (nch > p.max_chunks) {
        if (tid == 0) record_error(p.status, kDevBadSeqlens, 210);
        return;
    }
    if (k == 0) {  // only the window is kept
        if (tid == 0) {
            info[0] = -1;  // key 0xffffffff: no key is above it
            info[1] = -1;
        }
        for (int c = tid; c < nch; c += kThThreads) coff[c] = 0;
        return;
    }
    const float* pooled = p.pooled + static_cast<size_t>(u.g) * p.T + u.t0;
    for (int c = tid; c < nch; c += kThThreads) {
        cnt[c] = 0;
        eqc[c] = 0;
    }
    if (tid == 0) st.n_cand = 0;
    __syncthreads();
    find_digit(st.hist, k, st.scratch, &st.digit, &st.above);
    const uint32_t d1 = static_cast<uint32_t>(st.digit);
    const int r1 = k - st.above;           // rank of the k-th key within its first-digit bin
    const int bin_count = st.hist[d1];
    uint32_t thr;
    int pos_cut;
    if (bin_count <= kCandCap) {
        // One pass over the keys: count the keys of higher bins per chunk (all kept) and
        // collect the keys of bin d1 with their positions; the rest works in shared memory.
        for (int j0 = 0; j0 < P; j0 += 4 * kThThreads) {
            uint32_t key[4];
#pragma unroll
            for (int q = 0; q < 4; ++q) {
                const int j = j0 + q * kThThreads + tid;
                key[q] = j < P ? rank_key(__ldcg(pooled + j)) : 0u;
            }
#pragma unroll
            for (int q = 0; q < 4; ++q) {
                const int j = j0 + q * kThThreads + tid;  // a warp's 32 positions share a chunk
                const uint32_t b = key[q] >> kHistShift;
                const unsigned ba = __ballot_sync(0xffffffffu, j < P && b > d1);
                const unsigned bc = __ballot_sync(0xffffffffu, j < P && b == d1);
                if (lane == 0 && ba) atomicAdd(&cnt[(j0 + q * kThThreads + (tid & ~31)) >> kChunkShift], __popc(ba));
                if (bc) {
                    int slot = 0;
                    if (lane == 0) slot = atomicAdd(&st.n_cand, __popc(bc));
                    slot = __shfl_sync(0xffffffffu, slot, 0) + __popc(bc & ((1u << lane) - 1u));
                    if (((bc >> lane) & 1u) && slot < kCandCap) {
                        cand_key[slot] = key[q];
                        cand_pos[slot] = j;
                    }
                }
            }
        }
        __syncthreads();
        const int n = st.n_cand;
        if (n != bin_count) {  // the keys changed between the two reads
            if (tid == 0) record_error(p.status, kDevBadIndex, 310 + unit);
            return;
        }
        int need_eq, n_eq;
        thr = smem_select(cand_key, n, d1 << kHistShift, 0x7FFu << kHistShift, kHistShift, r1, st,
                          &need_eq, &n_eq);
        // mark the candidates: above the threshold, tied with it (by position), or dropped
        for (int i = tid; i < n; i += kThThreads) {
            const uint32_t x = cand_key[i];
            cand_key[i] = x > thr ? kTaken : (x == thr ? 0x7FFFFFFFu - static_cast<uint32_t>(cand_pos[i]) : kDropped);
        }
        __syncthreads();
        pos_cut = INT_MAX;  // every tie is kept
        if (need_eq < n_eq) {  // the need_eq-th smallest tie position, as the largest 0x7fffffff - pos
            int r_eq, n_eq2;
            const uint32_t v = smem_select(cand_key, n, 0u, 0x80000000u, 31, need_eq, st, &r_eq, &n_eq2);
            pos_cut = static_cast<int>(0x7FFFFFFFu - v);
        }
        for (int i = tid; i < n; i += kThThreads) {
            const uint32_t x = cand_key[i];
            if (x == kTaken || (x < 0x80000000u && static_cast<int>(0x7FFFFFFFu - x) <= pos_cut))
                atomicAdd(&cnt[cand_pos[i] >> kChunkShift], 1);
        }
        __syncthreads();
    } else {
        // Too many keys share the first digit: two more digit passes over all of the unit's
        // keys, then per-chunk counts of the keys above and equal to the threshold.
        uint32_t prefix = d1 << kHistShift, mask = 0x7FFu << kHistShift;
        int r = r1, last = 0;
#pragma unroll 1
        for (int level = 0; level < 2; ++level) {
            const int shift = level == 0 ? 10 : 0;
            const uint32_t dmask = level == 0 ? 0x7FFu : 0x3FFu;
            for (int b = tid; b < kHistBins; b += kThThreads) st.hist[b] = 0;
            __syncthreads();
            for (int j0 = 0; j0 < P; j0 += 4 * kThThreads) {
                uint32_t key[4];
#pragma unroll
                for (int q = 0; q < 4; ++q) {
                    const int j = j0 + q * kThThreads + tid;
                    key[q] = j < P ? rank_key(__ldcg(pooled + j)) : 0u;
                }
#pragma unroll
                for (int q = 0; q < 4; ++q) {
                    const int j = j0 + q * kThThreads + tid;
                    const bool in = j < P && (key[q] & mask) == prefix;
                    const uint32_t bin = in ? ((key[q] >> shift) & dmask) : static_cast<uint32_t>(kHistBins);
                    const unsigned peers = __match_any_sync(0xffffffffu, bin);
                    if (in && lane == __ffs(peers) - 1) atomicAdd(&st.hist[bin], __popc(peers));
                }
            }
            __syncthreads();
            find_digit(st.hist, r, st.scratch, &st.digit, &st.above);
            last = st.hist[st.digit];
            prefix |= static_cast<uint32_t>(st.digit) << shift;
            mask |= dmask << shift;
            r -= st.above;
            __syncthreads();
        }
        thr = prefix;
        const int need_eq = r, n_eq = last;
        for (int j0 = 0; j0 < P; j0 += 4 * kThThreads) {
            uint32_t key[4];
#pragma unroll
            for (int q = 0; q < 4; ++q) {
                const int j = j0 + q * kThThreads + tid;
                key[q] = j < P ? rank_key(__ldcg(pooled + j)) : 0u;
            }
#pragma unroll
            for (int q = 0; q < 4; ++q) {
                const int j = j0 + q * kThThreads + tid;
                const unsigned bg = __ballot_sync(0xffffffffu, j < P && key[q] > thr);
                const unsigned be = __ballot_sync(0xffffffffu, j < P && key[q] == thr);
                if (lane == 0 && (bg | be)) {
                    const int c = (j0 + q * kThThreads + (tid & ~31)) >> kChunkShift;
                    if (bg) atomicAdd(&cnt[c], __popc(bg));
                    if (be) atomicAdd(&eqc[c], __popc(be));
                }
            }
        }
        __syncthreads();
        pos_cut = INT_MAX;
        if (need_eq < n_eq) {
            // the chunk holding the need_eq-th tie in position order, then a walk through it
            if (tid == 0) {
                int before = 0, cc = nch - 1;
                for (int c = 0; c < nch; ++c) {
                    if (before + eqc[c] >= need_eq) {
                        cc = c;
                        break;
                    }
                    before += eqc[c];
                }
                st.cut_chunk = cc;
                st.cut_take = need_eq - before;
                st.cut_pos = INT_MAX;
            }
            __syncthreads();
            const int cc = st.cut_chunk, take = st.cut_take;
            int seen = 0;
            for (int b0 = cc * kChunk; b0 < min(P, (cc + 1) * kChunk); b0 += kThThreads) {
                const int j = b0 + tid;
                const bool is_eq = j < P && rank_key(__ldcg(pooled + j)) == thr;
                int tot;
                const int rk = block_excl_scan<kThThreads>(is_eq ? 1 : 0, st.scratch, &tot);
                if (is_eq && seen + rk == take - 1) st.cut_pos = j;
                seen += tot;
                if (seen >= take) break;  // uniform: every thread has the same `seen`
            }
            __syncthreads();
            pos_cut = st.cut_pos;
            for (int c = tid; c < nch; c += kThThreads)
                cnt[c] += c < cc ? eqc[c] : (c == cc ? take : 0);
        } else {
            for (int c = tid; c < nch; c += kThThreads) cnt[c] += eqc[c];
        }
        __syncthreads();
    }
    // output offsets of the chunks: an exclusive scan of their kept counts
    int carry = 0;
    for (int c0 = 0; c0 < nch; c0 += kThThreads) {
        const int c = c0 + tid;
        int tot;
        const int r = block_excl_scan<kThThreads>(c < nch ? cnt[c] : 0, st.scratch, &tot);
        if (c < nch) coff[c] = carry + r;
        carry += tot;
    }
    if (tid == 0) {
        info[0] = static_cast<int>(thr);
        info[1] = pos_cut;
        if (carry != k) record_error(p.status, kDevBadIndex, 300 + unit);
    }
}

__global__ void __launch_bounds__(kPHThreads) compact_kernel(const __grid_constant__ SelectParams p) {
    extern __shared__ int list[];  // [kChunk] the chunk's kept positions, in order
    __shared__ int wbase[kPHWarps + 1];
    const int unit = blockIdx.x, c = blockIdx.y, tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    if (unit == 0 && c == 0 && tid == 0 && seqlens_hash(p.cu_seqlens, p.S) != p.cu_hash)
        record_error(p.status, kDevBadSeqlens, 220);
    UnitGeo u;
    if (!unit_geo(p, unit, u)) return;
    if (u.g == 0 && c == 0 && tid == 0) {
        p.cu_keep[u.s + 1] = u.keep_off + u.n_keep;
        if (u.s == 0) p.cu_keep[0] = 0;
    }
    int32_t* out = p.idx + static_cast<size_t>(u.g) * p.T_keep + u.keep_off;
    const int j0 = c * kChunk;
    if (u.L <= p.budget) {  // kept whole
        const int m = max(0, min(u.L, j0 + kChunk) - j0);
        for (int e = tid; e < m; e += kPHThreads) {
            out[j0 + e] = j0 + e;
            list[e] = j0 + e;
        }
        __syncthreads();
        if (p.k) copy_rows(p, u, list, m, u.keep_off + j0);
        return;
    }
    const int P = u.P, k = u.k;
    if (c == 0) {  // the window closes the list
        for (int i = tid; i < p.w; i += kPHThreads) {
            out[k + i] = P + i;
            list[i] = P + i;
        }
        __syncthreads();
        if (p.k) copy_rows(p, u, list, p.w, u.keep_off + k);
        __syncthreads();
    }
    if (j0 >= P) return;
    const uint32_t thr = static_cast<uint32_t>(p.info[unit * 4]);
    const int pos_cut = p.info[unit * 4 + 1];
    const int base = p.chunk_off[static_cast<size_t>(unit) * p.max_chunks + c];
    const float* pooled = p.pooled + static_cast<size_t>(u.g) * p.T + u.t0;
    // warp w owns positions j0 + w*kWarpSpan ...: ballots give ranks in position order
    constexpr int kIt = kWarpSpan / 32;
    const int js = j0 + warp * kWarpSpan + lane;
    uint32_t key[kIt];
#pragma unroll
    for (int q = 0; q < kIt; ++q) {
        const int j = js + q * 32;
        key[q] = j < P ? rank_key(__ldcg(pooled + j)) : 0u;
    }
    unsigned bal[kIt];
    int wtot = 0;
#pragma unroll
    for (int q = 0; q < kIt; ++q) {
        const int j = js + q * 32;
        bal[q] = __ballot_sync(0xffffffffu, j < P && (key[q] > thr || (key[q] == thr && j <= pos_cut)));
        wtot += __popc(bal[q]);
    }
    if (lane == 0) wbase[warp] = wtot;
    __syncthreads();
    if (tid == 0) {
        int a = 0;
        for (int x = 0; x < kPHWarps; ++x) {
            const int t = wbase[x];
            wbase[x] = a;
            a += t;
        }
        wbase[kPHWarps] = a;
    }
    __syncthreads();
    const int tot = wbase[kPHWarps];
    if (base < 0 || base + tot > k) {
        if (tid == 0) record_error(p.status, kDevBadIndex, 320 + unit);
        return;
    }
    int r = wbase[warp];
    const unsigned lt = (1u << lane) - 1u;
#pragma unroll
    for (int q = 0; q < kIt; ++q) {
        if ((bal[q] >> lane) & 1u) {
            const int e = r + __popc(bal[q] & lt);
            out[base + e] = js + q * 32;
            list[e] = js + q * 32;
        }
        r += __popc(bal[q]);
    }
    __syncthreads();
    if (p.k) copy_rows(p, u, list, tot, u.keep_off + base);
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
    static SelectParams p;  // ~600 B; calls are serialised by `mu`
    static std::mutex mu;
    std::lock_guard<std::mutex> lock(mu);
    memset(&p, 0, sizeof p);
    p.scores = L.scores;
    p.pooled = L.pooled;
    p.idx = L.idx;
    p.cu_keep = L.cu_keep_dev;
    p.cu_seqlens = L.cu_seqlens_dev;
    p.status = L.status;
    p.hist = L.hist;
    p.info = L.info;
    p.chunk_off = L.chunk_off;
    p.k = reinterpret_cast<const uint4*>(L.k);
    p.v = reinterpret_cast<const uint4*>(L.v);
    p.tok_stride = L.tok_stride / 8;
    p.head_stride = L.head_stride / 8;
    p.k_out = reinterpret_cast<uint4*>(L.k_out);
    p.v_out = reinterpret_cast<uint4*>(L.v_out);
    p.S = L.S;
    p.T = L.T;
    p.Hkv = L.Hkv;
    p.w = L.w;
    p.budget = L.budget;
    p.T_keep = L.T_keep;
    p.max_chunks = L.max_chunks;
    p.pool_kernel = L.pool_kernel;
    p.pool_type = L.pool_type;
    p.head_order = L.head_order;
    p.from_scores = L.from_scores;
    p.write_pooled = L.write_pooled;
    p.cu_hash = L.cu_hash;
    for (int g = 0; g <= L.Hkv; ++g) p.group_first[g] = static_cast<int16_t>(L.group_first[g]);
    const int units = L.S * L.Hkv;
    if (units == 0 || L.max_chunks == 0) return cudaSuccess;
    if (L.max_chunks > 65535) return cudaErrorInvalidConfiguration;
    const size_t th_smem = sizeof(uint32_t) * 2 * kCandCap + sizeof(int) * 2 * static_cast<size_t>(L.max_chunks);
    static size_t th_smem_set = 0;
    static bool configured = false;
    cudaError_t e;
    if (!configured) {
        e = cudaFuncSetAttribute(pool_hist_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, kStageFloats * 4);
        if (e != cudaSuccess) return e;
        e = cudaFuncSetAttribute(compact_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, kCompactSmem);
        if (e != cudaSuccess) return e;
        configured = true;
    }
    if (th_smem > th_smem_set) {
        e = cudaFuncSetAttribute(threshold_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                 static_cast<int>(th_smem));
        if (e != cudaSuccess) return e;
        th_smem_set = th_smem;
    }
    const dim3 grid(units, L.max_chunks);
    pool_hist_kernel<<<grid, kPHThreads, kStageFloats * 4, stream>>>(p);
    if ((e = cudaGetLastError()) != cudaSuccess) return e;
    threshold_kernel<<<units, kThThreads, th_smem, stream>>>(p);
    if ((e = cudaGetLastError()) != cudaSuccess) return e;
    compact_kernel<<<grid, kPHThreads, kCompactSmem, stream>>>(p);
    return cudaGetLastError();
}

int select_chunks(int max_len) { return max(1, (max_len + kChunk - 1) / kChunk); }
size_t select_hist_ints() { return kHistBins; }

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
