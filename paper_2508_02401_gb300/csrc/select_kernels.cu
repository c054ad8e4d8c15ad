// Pooling, top-N selection and the K/V gather (arxiv 2508.02401, Sec. 3.3 and Fig. 3): the
// window-summed scores are smoothed along the token axis, the selected heads' vectors of a KV
// group are combined, the N best-scoring positions are kept and their K/V rows are copied
// into the compacted cache.
#include "ckv_device.cuh"
#include "ckv_internal.h"

#include <limits.h>
#include <string.h>

#include <algorithm>
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
// Per (sequence, KV head) unit: pool the scores (or read given pooled scores), take the k
// largest as order-preserving keys (ties: lowest positions first, as a stable sort by
// descending score keeps them), write their positions in position order followed by the
// window, and copy their K/V rows into the compacted cache when asked.
//
// Units of up to kUnitLen tokens are done by one 1024-thread block each (select_unit_kernel):
// every key stays in a register, and the k-th largest is found digit by digit (11, 11 and 10
// bits) with shared-memory counts.
//
// Longer units are cut into chunks of kChunk positions:
//   select_kernel  grid (unit, chunk): pools the chunk, counts its keys by their first digit
//                  into the unit's histogram and stores them grouped by that digit, highest
//                  first.  The last chunk block of a unit to finish gathers the keys of the
//                  digit that holds the k-th largest from every chunk's group and finds the
//                  threshold key, the tie cutoff position and each chunk's output offset.
//   compact_kernel grid (unit, chunk): writes the chunk's kept positions in position order and
//                  copies their rows; chunk 0 also writes the window.
// The unit histograms and arrival counters are zero outside a call: the last block of each
// unit clears them once it has read them.
constexpr int kChunk = 4096;                 // candidate positions per chunk
constexpr int kChunkShift = 12;
constexpr int kHistBins = 2048;              // digits of up to 11 bits
constexpr int kHistShift = 21;               // the first digit is bits 31..21 of a key
constexpr int kSelThreads = 512;             // select_kernel and compact_kernel
constexpr int kSelWarps = kSelThreads / 32;
constexpr int kPHPer = kChunk / kSelThreads; // contiguous positions per thread
constexpr int kWarpSpan = kChunk / kSelWarps; // compact: contiguous positions per warp
constexpr int kMaxHalo = kMaxPoolKernel / 2;
constexpr int kStageFloats = kChunk + 2 * kMaxHalo;
constexpr int kStageLoads = (kStageFloats + kSelThreads - 1) / kSelThreads;
constexpr int kCandCap = 8192;               // candidates held in shared memory
constexpr int kTieCap = 256;                 // ties ranked pairwise up to this many
constexpr int kCompactSmem = kChunk * 4;     // compact: the chunk's kept positions
constexpr uint32_t kTaken = 0xFFFFFFFEu;     // tie-select markers; the top bit keeps both out
constexpr uint32_t kDropped = 0xFFFFFFFFu;   //   of the position select
constexpr int kUnitThreads = 1024;           // select_unit_kernel
constexpr int kUnitPer = 16;
constexpr int kUnitLen = kUnitThreads * kUnitPer;
constexpr int kUnitStage = kUnitLen + 2 * kMaxHalo;
constexpr int kUnitStageLoads = (kUnitStage + kUnitThreads - 1) / kUnitThreads;
constexpr int kUnitCandMax = 1024;            // first-digit ties ranked pairwise up to this many
static_assert(kWarpSpan % 32 == 0 && (1 << kChunkShift) == kChunk, "chunk shape");

// Shared-memory index of staged element e: one pad word per 32 keeps the contiguous
// per-thread reads of the pooling free of bank conflicts.
__device__ __forceinline__ int sidx(int e) { return e + (e >> 5); }
constexpr int stage_words(int n) { return n + (n >> 5) + 2; }
constexpr int kUnitSmem = stage_words(kUnitStage) * 4;
constexpr int kSelStageSmem = stage_words(kStageFloats) * 4;

struct SelectParams {
    const float* scores;   // [n_sel, T]: pooled here when from_scores != 0
    float* pooled;         // [H_kv, T]
    int32_t* idx;          // [H_kv, T_keep]
    int32_t* cu_keep;      // [S+1]
    const int32_t* cu_seqlens;
    int* status;
    int* hist;             // [units][kHistBins] first-digit counts
    int* arrivals;         // [units] chunk blocks done
    int* chunk_start;      // [units][max_chunks][kHistBins] start of each digit group
    uint2* buckets;        // [units][max_chunks][kChunk] (key, position) grouped by digit
    int* info;             // [units][4]: threshold key, tie cutoff position
    int* chunk_off;        // [units][max_chunks]: output offset of each chunk's kept positions
    const uint4* k;        // gather source (nullptr: no gather); strides in 16-byte units
    const uint4* v;
    int64_t tok_stride, head_stride;
    uint4* k_out;
    uint4* v_out;
    int S, T, Hkv, w, budget, T_keep, max_chunks;
    int n_vec;             // selections per sequence: H_kv (per KV head) or 1 (per layer)
    int pool_kernel, pool_type, head_order, from_scores, write_pooled;
    uint32_t cu_hash;
    int16_t group_first[kMaxQHeads + 1];
};

__device__ __forceinline__ int atomic_add_acq_rel(int* p, int v) {
    int old;
    asm volatile("atom.acq_rel.gpu.global.add.s32 %0, [%1], %2;" : "=r"(old) : "l"(p), "r"(v) : "memory");
    return old;
}

// Order-preserving unsigned key of a float (-0 and +0 share one key).
__device__ __forceinline__ uint32_t rank_key(float f) {
    uint32_t u = __float_as_uint(f);
    if (u == 0x80000000u) u = 0u;
    return (u & 0x80000000u) ? ~u : (u | 0x80000000u);
}

struct UnitGeo {
    int s, g, t0, L, P, k, keep_off, n_keep;  // g: the selection (KV head, or 0 per layer)
};

// Geometry of unit (sequence s, KV head g), from the device cu_seqlens; false (and an error
// recorded) if they are unusable.  Every thread of the block calls it.
__device__ __forceinline__ bool unit_geo(const SelectParams& p, int unit, UnitGeo& u) {
    u.s = unit / p.n_vec;
    u.g = unit % p.n_vec;
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

// Block-wide exclusive prefix sum in thread order over NT threads; *total gets the sum.
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

// The same with one barrier: each warp's sum goes to buf[warp], then every warp adds up the
// sums of the warps before it.  Consecutive calls must alternate between two buffers: a call's
// barrier then orders every read of the buffer two calls back before it is written again.
template <int NT>
__device__ __forceinline__ int block_excl_scan1(int v, int* buf, int* total) {
    constexpr int NW = NT / 32;
    static_assert(NW <= 32, "warps");
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    int incl = v;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        const int y = __shfl_up_sync(0xffffffffu, incl, o);
        if (lane >= o) incl += y;
    }
    if (lane == 31) buf[warp] = incl;
    __syncthreads();
    const int x = lane < NW ? buf[lane] : 0;
    const int before = __reduce_add_sync(0xffffffffu, lane < warp ? x : 0);
    *total = __reduce_add_sync(0xffffffffu, x);
    return before + incl - v;
}

// The digit d of a kHistBins-bin histogram with count(bins above d) < r <= count(bins >= d),
// r >= 1: *s_digit = d, *s_above = count(bins above d).  Thread 0 owns the highest bins.
template <int NT>
__device__ __forceinline__ void find_digit(const int* hist, int r, int* scratch, int* s_digit,
                                           int* s_above) {
    constexpr int PER = kHistBins / NT;
    if (threadIdx.x == 0) {
        *s_digit = 0;
        *s_above = 0;
    }
    const int base = (NT - 1 - static_cast<int>(threadIdx.x)) * PER;
    int local = 0;
#pragma unroll
    for (int q = 0; q < PER; ++q) local += hist[base + q];
    int tot;
    const int above = block_excl_scan<NT>(local, scratch, &tot);
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

// Adds a thread's run-aggregated counts of PER consecutive digits (v[i] >> SHIFT) to a shared
// histogram: consecutive keys of a thread are neighbouring positions and often share a digit,
// so one atomic add per run of equal digits (a linear scan) instead of one per key.  Digits
// below `lo` are not counted.
template <int PER, int SHIFT = 0>
__device__ __forceinline__ void add_runs(int* hist, const uint32_t (&v)[PER], int nvalid, uint32_t lo = 0) {
    if (nvalid <= 0) return;
    uint32_t cur = v[0] >> SHIFT;
    int len = 1;
#pragma unroll
    for (int i = 1; i < PER; ++i) {
        if (i < nvalid) {
            const uint32_t d = v[i] >> SHIFT;
            if (d == cur) {
                ++len;
            } else {
                if (cur >= lo) atomicAdd(&hist[cur], len);
                cur = d;
                len = 1;
            }
        }
    }
    if (cur >= lo) atomicAdd(&hist[cur], len);
}

// Stages the sum of score rows [ra, rb) at sequence positions base-half .. base+n+half-1
// (zero outside [0, P)) into st, element e at st[sidx(e)]; loads are coalesced and all of a
// row's loads of a thread are issued before its stores.
template <int NT, int LOADS>
__device__ __forceinline__ void stage_rows(float* st, const float* scores, size_t T, int t0, int ra,
                                           int rb, int base, int half, int n, int P) {
    const int ne = n + 2 * half, tid = threadIdx.x;
    float xs[LOADS];
#pragma unroll
    for (int i = 0; i < LOADS; ++i) xs[i] = 0.f;
    for (int r = ra; r < rb; ++r) {
        const float* row = scores + static_cast<size_t>(r) * T + t0;
#pragma unroll
        for (int i = 0; i < LOADS; ++i) {
            const int e = tid + i * NT;
            const int uu = base - half + e;
            if (e < ne && uu >= 0 && uu < P) xs[i] += __ldg(row + uu);
        }
    }
#pragma unroll
    for (int i = 0; i < LOADS; ++i) {
        const int e = tid + i * NT;
        if (e < ne) st[sidx(e)] = xs[i];
    }
}

__device__ __forceinline__ void cp_async4(float* dst, const float* src) {
    asm volatile("cp.async.ca.shared.global [%0], [%1], 4;" ::"r"(smem_u32(dst)), "l"(src) : "memory");
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }
template <int N>
__device__ __forceinline__ void cp_async_wait_group() {
    asm volatile("cp.async.wait_group %0;" ::"n"(N) : "memory");
}

// Issues the copies that stage score rows ra .. ra+nr-1 (each alone, not summed) at sequence
// positions base-half .. base+n+half-1 (zero outside [0, P)), row i at st + i*words, element e
// at sidx(e), and commits them as one group: every copy of every row is issued
// (asynchronously, no registers held) before any wait, so the rows take one round trip together.
template <int NT, int LOADS>
__device__ __forceinline__ void stage_rows_issue(float* st, int words, const float* scores, size_t T,
                                                 int t0, int ra, int nr, int base, int half, int n,
                                                 int P) {
    const int ne = n + 2 * half, tid = threadIdx.x;
    for (int i = 0; i < nr; ++i) {
        const float* row = scores + static_cast<size_t>(ra + i) * T + t0;
        float* dst = st + i * words;
#pragma unroll
        for (int q = 0; q < LOADS; ++q) {
            const int e = tid + q * NT;
            const int uu = base - half + e;
            if (e < ne) {
                if (uu >= 0 && uu < P) cp_async4(dst + sidx(e), row + uu);
                else dst[sidx(e)] = 0.f;
            }
        }
    }
    cp_async_commit();
}

// The same, waiting for this thread's copies to land.
template <int NT, int LOADS>
__device__ __forceinline__ void stage_rows_async(float* st, int words, const float* scores, size_t T,
                                                 int t0, int ra, int nr, int base, int half, int n,
                                                 int P) {
    stage_rows_issue<NT, LOADS>(st, words, scores, T, t0, ra, nr, base, half, n, P);
    cp_async_wait_group<0>();
}

// Pools PER consecutive outputs from the stage: output i reads staged elements
// jl+i .. jl+i+2*HALF.  Same arithmetic, in the same order, as pool_kernel: the staged zeros
// outside [0, P) leave a max of non-negative scores and a left-to-right sum unchanged.
template <int HALF, int PER>
__device__ __forceinline__ void pool_window(const float* st, int jl, int nvalid, bool is_max, float kf,
                                            float (&acc)[PER]) {
    float w[PER + 2 * HALF];
#pragma unroll
    for (int i = 0; i < PER + 2 * HALF; ++i) w[i] = st[sidx(jl + i)];
#pragma unroll
    for (int i = 0; i < PER; ++i) {
        if (i < nvalid) {
            float m = w[i];
            if (is_max) {
#pragma unroll
                for (int t = 1; t <= 2 * HALF; ++t) m = fmaxf(m, w[i + t]);
                acc[i] += m;
            } else {
#pragma unroll
                for (int t = 1; t <= 2 * HALF; ++t) m += w[i + t];
                acc[i] += m / kf;  // IEEE division, as in pool_kernel
            }
        }
    }
}

template <int PER>
__device__ __forceinline__ void pool_any(const float* st, int jl, int nvalid, int half, bool is_max,
                                         float kf, float (&acc)[PER]) {
    // A thread with no output reads nothing: its window would start past the staged row (and,
    // for the last of several staged rows, past the stage).  A thread with outputs reads at most
    // PER - 1 elements past its row's last staged one.
    if (nvalid <= 0) return;
    if (half == 3) {
        pool_window<3, PER>(st, jl, nvalid, is_max, kf, acc);
    } else if (half == 2) {
        pool_window<2, PER>(st, jl, nvalid, is_max, kf, acc);
    } else {
#pragma unroll
        for (int i = 0; i < PER; ++i) {
            if (i < nvalid) {
                float m = st[sidx(jl + i)];
                for (int t = 1; t <= 2 * half; ++t)
                    m = is_max ? fmaxf(m, st[sidx(jl + i + t)]) : m + st[sidx(jl + i + t)];
                acc[i] += is_max ? m : m / kf;
            }
        }
    }
}

// Pooled scores of positions base+jl .. base+jl+PER-1 (jl = PER * thread) of unit u, computed
// from the scores (from_scores) or read from p.pooled.  Ends with the stage free again.
// WORDS is the stage's capacity: with the heads pooled one by one, as many rows as fit are
// staged together.
template <int NT, int PER, int LOADS, int WORDS>
__device__ __forceinline__ void pooled_values(const SelectParams& p, const UnitGeo& u, float* st, int base,
                                              int n, float (&acc)[PER]) {
    const int jl = threadIdx.x * PER, nvalid = n - jl;
#pragma unroll
    for (int i = 0; i < PER; ++i) acc[i] = 0.f;
    if (p.from_scores) {
        const int half = p.pool_kernel >> 1;
        const bool is_max = p.pool_type == 0;
        const float kf = static_cast<float>(p.pool_kernel);
        const int r0 = p.group_first[u.g], r1 = p.group_first[u.g + 1];
        if (p.head_order == 0) {  // pool each head, then sum (in head order)
            const int words = stage_words(n + 2 * half);
            // rows that fit, with room for the last row's readers to run PER words past it
            const int fit = max(1, (WORDS - PER) / words);
            for (int ra = r0; ra < r1; ra += fit) {
                const int nr = min(fit, r1 - ra);
                stage_rows_async<NT, LOADS>(st, words, p.scores, p.T, u.t0, ra, nr, base, half, n, u.P);
                __syncthreads();
                for (int i = 0; i < nr; ++i) pool_any<PER>(st + i * words, jl, nvalid, half, is_max, kf, acc);
                __syncthreads();
            }
        } else {  // sum the heads, then pool
            stage_rows<NT, LOADS>(st, p.scores, p.T, u.t0, r0, r1, base, half, n, u.P);
            __syncthreads();
            pool_any<PER>(st, jl, nvalid, half, is_max, kf, acc);
            __syncthreads();
        }
    } else {
        const float* src = p.pooled + static_cast<size_t>(u.g) * p.T + u.t0 + base;
#pragma unroll
        for (int i = 0; i < LOADS; ++i) {
            const int e = threadIdx.x + i * NT;
            if (e < n) st[sidx(e)] = __ldg(src + e);
        }
        __syncthreads();
#pragma unroll
        for (int i = 0; i < PER; ++i)
            if (i < nvalid) acc[i] = st[sidx(jl + i)];
        __syncthreads();
    }
}

// Copies the K and V rows of sequence-local positions list[0..m) to output rows
// out_row0 + 0..m-1 of KV head g: a warp per row (16 lanes for K, 16 for V), kRowsInFlight
// rows in flight per warp (not inlined: the rows in flight then stay in registers whatever the
// caller holds).
constexpr int kRowsInFlight = 8;
__device__ __noinline__ void copy_rows(const SelectParams& p, const UnitGeo& u, int kv,
                                          const int* list, int m, int out_row0) {
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31, nw = blockDim.x >> 5;
    const int part = lane & 15;
    const uint4* src0 = (lane < 16 ? p.k : p.v) + static_cast<int64_t>(u.t0) * p.tok_stride +
                        static_cast<int64_t>(kv) * p.head_stride + part;
    uint4* dst0 = (lane < 16 ? p.k_out : p.v_out) + static_cast<int64_t>(kv) * 16 + part;
    for (int e0 = warp; e0 < m; e0 += kRowsInFlight * nw) {
        uint4 x[kRowsInFlight];
#pragma unroll
        for (int q = 0; q < kRowsInFlight; ++q) {
            const int e = e0 + q * nw;
            if (e < m) x[q] = __ldg(src0 + static_cast<int64_t>(list[e]) * p.tok_stride);
        }
#pragma unroll
        for (int q = 0; q < kRowsInFlight; ++q) {
            const int e = e0 + q * nw;
            if (e < m) dst0[static_cast<int64_t>(out_row0 + e) * p.Hkv * 16] = x[q];
        }
    }
}

// Writes list[0..m) (sequence-local positions, in order) to the index rows at offset out_off
// of the unit's kept tokens, and copies the K/V rows when asked, for KV heads [kv0, kv1) of
// those the unit's selection serves: its own (per-KV-head scope) or all of them (per-layer
// scope).
__device__ __forceinline__ void emit_kept(const SelectParams& p, const UnitGeo& u, const int* list,
                                          int m, int out_off, int kv0, int kv1) {
    for (int kv = kv0; kv < kv1; ++kv) {
        int32_t* out = p.idx + static_cast<size_t>(kv) * p.T_keep + u.keep_off + out_off;
        for (int e = threadIdx.x; e < m; e += blockDim.x) out[e] = list[e];
        if (p.k) copy_rows(p, u, kv, list, m, u.keep_off + out_off);
    }
}

// ------------------------------------------------------------------ units of up to kUnitLen
__global__ void __launch_bounds__(kUnitThreads, 1) select_unit_kernel(const __grid_constant__ SelectParams p) {
    extern __shared__ __align__(16) float ust[];  // pooling stage, then the kept list
    __shared__ int hist[kHistBins];
    __shared__ int scratch[33];
    __shared__ int s_digit, s_above, s_cut, s_cnt;
    __shared__ uint32_t s_thr;
    constexpr int NT = kUnitThreads, PER = kUnitPer;
    // A selection that serves several KV heads (per-layer scope) is made by one block per KV
    // head, each gathering its own head's rows: the selection is recomputed (from L2-resident
    // scores) rather than one block copying every head's rows alone.
    const int per = p.Hkv / p.n_vec;
    const int unit = blockIdx.x / per, sub = blockIdx.x % per, tid = threadIdx.x;
    if (blockIdx.x == 0 && tid == 0 && seqlens_hash(p.cu_seqlens, p.S) != p.cu_hash)
        record_error(p.status, kDevBadSeqlens, 230);
    UnitGeo u;
    if (!unit_geo(p, unit, u)) return;
    if (u.L > kUnitLen) return;  // a long unit: the chunked kernels take it
    const int kv = u.g * per + sub;  // the KV head whose rows this block writes
    if (u.g == 0 && sub == 0 && tid == 0) {
        p.cu_keep[u.s + 1] = u.keep_off + u.n_keep;
        if (u.s == 0) p.cu_keep[0] = 0;
    }
    float* pooled = p.pooled + static_cast<size_t>(u.g) * p.T + u.t0;
    int* list = reinterpret_cast<int*>(ust);
    const bool zeros = p.from_scores && p.write_pooled && sub == 0;
    if (u.L <= p.budget) {  // kept whole; its pooled scores read as 0
        for (int e = tid; e < u.L; e += NT) {
            list[e] = e;
            if (zeros) pooled[e] = 0.f;
        }
        __syncthreads();
        emit_kept(p, u, list, u.L, 0, kv, kv + 1);
        return;
    }
    const int P = u.P, k = u.k;
    if (zeros)  // window positions are not candidates
        for (int j = P + tid; j < u.L; j += NT) pooled[j] = 0.f;
    const int jb = tid * PER, nvalid = P - jb;
    float acc[PER];
    pooled_values<NT, PER, kUnitStageLoads, stage_words(kUnitStage)>(p, u, ust, 0, P, acc);
    if (zeros)
#pragma unroll
        for (int i = 0; i < PER; ++i)
            if (i < nvalid) pooled[jb + i] = acc[i];
    uint32_t key[PER], bins[PER];
#pragma unroll
    for (int i = 0; i < PER; ++i) {
        key[i] = rank_key(acc[i]);
        bins[i] = key[i] >> kHistShift;
    }
    // the k-th largest key, digit by digit (k = 0 keeps only the window: no key is above
    // 0xffffffff and no position is at or below -1)
    uint32_t thr = 0xFFFFFFFFu;
    int pos_cut = -1;
    if (k > 0) {
        for (int b = tid; b < kHistBins; b += NT) hist[b] = 0;
        if (tid == 0) s_cut = INT_MAX;
        __syncthreads();
        add_runs<PER>(hist, bins, nvalid);
        __syncthreads();
        find_digit<NT>(hist, k, scratch, &s_digit, &s_above);
        uint32_t prefix = static_cast<uint32_t>(s_digit) << kHistShift, mask = 0x7FFu << kHistShift;
        int r = k - s_above, n_eq = hist[s_digit];
        __syncthreads();
        if (n_eq <= kUnitCandMax) {
            // Few keys share the k-th key's first digit: gather them and rank them exactly, by
            // key descending then position ascending; the r-th is the threshold key, its
            // position the tie cutoff.  (The stage is free again: it holds the pairs.)
            uint2* cand = reinterpret_cast<uint2*>(ust);
            const uint32_t d = static_cast<uint32_t>(s_digit);
            if (tid == 0) s_cnt = 0;
            __syncthreads();
#pragma unroll
            for (int i = 0; i < PER; ++i)
                if (i < nvalid && bins[i] == d) cand[atomicAdd(&s_cnt, 1)] = make_uint2(key[i], jb + i);
            __syncthreads();
            for (int c = tid; c < n_eq; c += NT) {
                const uint2 me = cand[c];
                int ahead = 0;
                for (int q = 0; q < n_eq; ++q) {
                    const uint2 o = cand[q];
                    ahead += (o.x > me.x || (o.x == me.x && o.y < me.y)) ? 1 : 0;
                }
                if (ahead == r - 1) {
                    s_thr = me.x;
                    s_cut = static_cast<int>(me.y);
                }
            }
            __syncthreads();
            thr = s_thr;
            pos_cut = s_cut;
        } else {
#pragma unroll 1
            for (int level = 0; level < 2; ++level) {
                const int shift = level == 0 ? 10 : 0;
                const uint32_t dmask = level == 0 ? 0x7FFu : 0x3FFu;
                for (int b = tid; b < kHistBins; b += NT) hist[b] = 0;
                __syncthreads();
#pragma unroll
                for (int i = 0; i < PER; ++i)
                    if (i < nvalid && (key[i] & mask) == prefix) atomicAdd(&hist[(key[i] >> shift) & dmask], 1);
                __syncthreads();
                find_digit<NT>(hist, r, scratch, &s_digit, &s_above);
                prefix |= static_cast<uint32_t>(s_digit) << shift;
                mask |= dmask << shift;
                r -= s_above;
                n_eq = hist[s_digit];
                __syncthreads();
            }
            thr = prefix;
            const int need_eq = r;  // keys equal to thr that are kept: the lowest positions
            pos_cut = INT_MAX;
            if (need_eq < n_eq) {
                int ne = 0;
#pragma unroll
                for (int i = 0; i < PER; ++i) ne += (i < nvalid && key[i] == thr) ? 1 : 0;
                int tot;
                const int before = block_excl_scan<NT>(ne, scratch, &tot);  // thread order = position order
                if (before < need_eq && before + ne >= need_eq) {
                    int c = before;
#pragma unroll
                    for (int i = 0; i < PER; ++i) {
                        if (i < nvalid && key[i] == thr) {
                            ++c;
                            if (c == need_eq) s_cut = jb + i;
                        }
                    }
                }
                __syncthreads();
                pos_cut = s_cut;
            }
        }
    }
    // the kept positions in order, then the window
    uint32_t taken = 0;
    int cnt = 0;
#pragma unroll
    for (int i = 0; i < PER; ++i) {
        if (i < nvalid && (key[i] > thr || (key[i] == thr && jb + i <= pos_cut))) {
            taken |= 1u << i;
            ++cnt;
        }
    }
    int tot;
    int rk = block_excl_scan<NT>(cnt, scratch, &tot);
    if (tot != k) {
        if (tid == 0) record_error(p.status, kDevBadIndex, 330 + unit);
        return;
    }
#pragma unroll
    for (int i = 0; i < PER; ++i) {
        if ((taken >> i) & 1u) {
            list[rk] = jb + i;
            ++rk;
        }
    }
    for (int i = tid; i < p.w; i += NT) list[k + i] = P + i;
    __syncthreads();
    emit_kept(p, u, list, p.budget, 0, kv, kv + 1);
}

// ------------------------------------------------------------------ longer units, in chunks
struct SelectShared {
    int hist[kHistBins];   // chunk counts, then group starts; the unit's counts in the last block
    int fill[kHistBins];   // group fill pointers
    int scratch[33];
    int digit, above, last, n_cand, n_tie, cut;
};

// The r-th largest (r >= 1) of the values get(0..n) whose bits under `mask` equal `prefix`,
// digit by digit over the `bits` lower bits.  *r_eq gets how many copies of the result rank
// within the first r, *n_eq how many copies there are.  Uses (and leaves garbage in) sh.hist.
template <class Get>
__device__ uint32_t radix_select(Get get, int n, uint32_t prefix, uint32_t mask, int bits, int r,
                                 SelectShared& sh, int* r_eq, int* n_eq) {
    const int tid = threadIdx.x, lane = tid & 31;
    int last = 0;
    while (bits > 0) {
        const int d = bits > 11 ? 11 : bits;
        const int shift = bits - d;
        const uint32_t dmask = (1u << d) - 1u;
        for (int b = tid; b < kHistBins; b += kSelThreads) sh.hist[b] = 0;
        __syncthreads();
        for (int i0 = 0; i0 < n; i0 += kSelThreads) {
            const int i = i0 + tid;
            const uint32_t x = i < n ? get(i) : 0u;
            const bool in = i < n && (x & mask) == prefix;
            if (__any_sync(0xffffffffu, in)) {
                const uint32_t bin = in ? (x >> shift) & dmask : static_cast<uint32_t>(kHistBins);
                const unsigned peers = __match_any_sync(0xffffffffu, bin);
                if (in && lane == __ffs(peers) - 1) atomicAdd(&sh.hist[bin], __popc(peers));
            }
        }
        __syncthreads();
        find_digit<kSelThreads>(sh.hist, r, sh.scratch, &sh.digit, &sh.above);
        const int dg = sh.digit;
        last = sh.hist[dg];
        prefix |= static_cast<uint32_t>(dg) << shift;
        mask |= dmask << shift;
        r -= sh.above;
        bits -= d;
        __syncthreads();  // hist and digit are read before the next digit reuses them
    }
    *r_eq = r;
    *n_eq = last;
    return prefix;
}

// The threshold of one unit, run by the last of its chunk blocks (see select_kernel).
// dyn: cand_key[kCandCap] cand_pos[kCandCap] above[max_chunks] coff[max_chunks+1] cnt[max_chunks]
//      tie_pos[kTieCap]
__device__ __noinline__ void unit_threshold(const SelectParams& p, const UnitGeo& u, int unit, int nch,
                                            SelectShared& sh, uint32_t* dyn) {
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    uint32_t* cand_key = dyn;
    int* cand_pos = reinterpret_cast<int*>(dyn + kCandCap);
    int* above = reinterpret_cast<int*>(dyn + 2 * kCandCap);
    int* coff = above + p.max_chunks;
    int* cnt = coff + p.max_chunks + 1;
    int* tie_pos = cnt + p.max_chunks;
    int* info = p.info + unit * 4;
    int* out_off = p.chunk_off + static_cast<size_t>(unit) * p.max_chunks;
    const int P = u.P, k = u.k;
    // the unit's digit counts, left zeroed for the next call
    int* gh = p.hist + static_cast<size_t>(unit) * kHistBins;
    for (int b = tid; b < kHistBins; b += kSelThreads) {
        sh.hist[b] = __ldcg(gh + b);
        __stcg(gh + b, 0);
    }
    if (tid == 0) {
        p.arrivals[unit] = 0;
        sh.n_tie = 0;
        sh.cut = INT_MAX;
    }
    __syncthreads();
    if (k == 0) {  // only the window is kept
        if (tid == 0) {
            info[0] = -1;  // key 0xffffffff: no key is above it
            info[1] = -1;
        }
        for (int c = tid; c < nch; c += kSelThreads) out_off[c] = 0;
        return;
    }
    find_digit<kSelThreads>(sh.hist, k, sh.scratch, &sh.digit, &sh.above);
    const uint32_t d1 = static_cast<uint32_t>(sh.digit);
    const int r1 = k - sh.above;  // rank of the k-th key among the keys of digit d1
    const int n = sh.hist[d1];
    // per chunk: keys of higher digits (all kept) and the group of digit d1
    const int* cs = p.chunk_start + static_cast<size_t>(unit) * p.max_chunks * kHistBins;
    int carry = 0;
    for (int c0 = 0; c0 < nch; c0 += kSelThreads) {
        const int c = c0 + tid;
        int m = 0;
        if (c < nch) {
            const int a = __ldcg(cs + static_cast<size_t>(c) * kHistBins + d1);
            const int e = d1 == 0 ? min(kChunk, P - c * kChunk)
                                  : __ldcg(cs + static_cast<size_t>(c) * kHistBins + d1 - 1);
            above[c] = a;
            m = e - a;
        }
        int tot;
        const int r = block_excl_scan<kSelThreads>(m, sh.scratch, &tot);
        if (c < nch) coff[c] = carry + r;
        carry += tot;
    }
    if (tid == 0) coff[nch] = carry;
    __syncthreads();
    if (carry != n) {
        if (tid == 0) record_error(p.status, kDevBadIndex, 300 + unit);
        return;
    }
    const uint2* bk = p.buckets + static_cast<size_t>(unit) * p.max_chunks * kChunk;
    // candidate i: from shared memory, or found in its chunk's group when there are too many
    const bool in_smem = n <= kCandCap;
    if (in_smem) {
        for (int c = warp; c < nch; c += kSelWarps) {
            const int a = above[c], o = coff[c], m = coff[c + 1] - o;
            for (int i = lane; i < m; i += 32) {
                const uint2 e = __ldcg(bk + static_cast<size_t>(c) * kChunk + a + i);
                cand_key[o + i] = e.x;
                cand_pos[o + i] = static_cast<int>(e.y);
            }
        }
        __syncthreads();
    }
    auto cand = [&](int i) -> uint2 {
        if (in_smem) return make_uint2(cand_key[i], static_cast<uint32_t>(cand_pos[i]));
        int lo = 0, hi = nch - 1;  // the chunk c with coff[c] <= i < coff[c+1]
        while (lo < hi) {
            const int mid = (lo + hi + 1) >> 1;
            if (coff[mid] <= i) lo = mid;
            else hi = mid - 1;
        }
        return __ldcg(bk + static_cast<size_t>(lo) * kChunk + above[lo] + (i - coff[lo]));
    };
    int need_eq, n_eq;
    const uint32_t thr = radix_select([&](int i) { return cand(i).x; }, n, d1 << kHistShift,
                                      0x7FFu << kHistShift, kHistShift, r1, sh, &need_eq, &n_eq);
    // Of the candidates equal to thr the need_eq lowest positions are kept: ranked pairwise
    // when there are few, else found as the need_eq-th largest 0x7fffffff - position.
    int pos_cut = INT_MAX;
    if (need_eq < n_eq) {
        if (n_eq <= kTieCap) {
            for (int i0 = 0; i0 < n; i0 += kSelThreads) {
                const int i = i0 + tid;
                const bool eq = i < n && cand(i).x == thr;
                const unsigned b = __ballot_sync(0xffffffffu, eq);
                if (b) {
                    int at = 0;
                    if (lane == 0) at = atomicAdd(&sh.n_tie, __popc(b));
                    at = __shfl_sync(0xffffffffu, at, 0) + __popc(b & ((1u << lane) - 1u));
                    if (eq) tie_pos[at] = static_cast<int>(cand(i).y);
                }
            }
            __syncthreads();
            if (tid < n_eq) {
                const int mine = tie_pos[tid];
                int rank = 0;
                for (int q = 0; q < n_eq; ++q) rank += tie_pos[q] < mine ? 1 : 0;
                if (rank == need_eq - 1) sh.cut = mine;
            }
        } else {
            auto mark = [&](int i) -> uint32_t {
                const uint2 e = cand(i);
                return e.x > thr ? kTaken : (e.x == thr ? 0x7FFFFFFFu - e.y : kDropped);
            };
            int r_eq, n_eq2;
            const uint32_t v = radix_select(mark, n, 0u, 0x80000000u, 31, need_eq, sh, &r_eq, &n_eq2);
            if (tid == 0) sh.cut = static_cast<int>(0x7FFFFFFFu - v);
        }
        __syncthreads();
        pos_cut = sh.cut;
    }
    for (int c = tid; c < nch; c += kSelThreads) cnt[c] = above[c];
    __syncthreads();
    for (int i = tid; i < n; i += kSelThreads) {
        const uint2 e = cand(i);
        if (e.x > thr || (e.x == thr && static_cast<int>(e.y) <= pos_cut))
            atomicAdd(&cnt[e.y >> kChunkShift], 1);
    }
    __syncthreads();
    carry = 0;
    for (int c0 = 0; c0 < nch; c0 += kSelThreads) {
        const int c = c0 + tid;
        int tot;
        const int r = block_excl_scan<kSelThreads>(c < nch ? cnt[c] : 0, sh.scratch, &tot);
        if (c < nch) out_off[c] = carry + r;
        carry += tot;
    }
    if (tid == 0) {
        info[0] = static_cast<int>(thr);
        info[1] = pos_cut;
        if (carry != k) record_error(p.status, kDevBadIndex, 310 + unit);
    }
}

__global__ void __launch_bounds__(kSelThreads) select_kernel(const __grid_constant__ SelectParams p) {
    extern __shared__ __align__(16) uint32_t dyn[];  // pooling stage, later the threshold's arrays
    __shared__ SelectShared sh;
    constexpr int PER = kPHPer;
    const int unit = blockIdx.x, c = blockIdx.y, tid = threadIdx.x;
    if (unit == 0 && c == 0 && tid == 0 && seqlens_hash(p.cu_seqlens, p.S) != p.cu_hash)
        record_error(p.status, kDevBadSeqlens, 200);
    UnitGeo u;
    if (!unit_geo(p, unit, u)) return;
    if (u.L <= kUnitLen) return;  // select_unit_kernel takes it
    float* pooled = p.pooled + static_cast<size_t>(u.g) * p.T + u.t0;
    const int j0 = c * kChunk;
    const bool zeros = p.from_scores && p.write_pooled;
    if (u.L <= p.budget) {  // kept whole: nothing to select; its pooled scores read as 0
        if (zeros)
            for (int j = j0 + tid; j < min(u.L, j0 + kChunk); j += kSelThreads) pooled[j] = 0.f;
        return;
    }
    const int nch = (u.P + kChunk - 1) / kChunk;
    if (nch > p.max_chunks) {  // longer than the host lengths said: leave the unit alone
        if (c == 0 && tid == 0) record_error(p.status, kDevBadSeqlens, 210);
        return;
    }
    if (zeros)  // window positions are not candidates
        for (int j = max(j0, u.P) + tid; j < min(u.L, j0 + kChunk); j += kSelThreads) pooled[j] = 0.f;
    if (j0 >= u.P) return;
    const int n = min(kChunk, u.P - j0);
    const int jl = tid * PER, nvalid = n - jl;
    float acc[PER];
    pooled_values<kSelThreads, PER, kStageLoads, stage_words(kStageFloats)>(p, u, reinterpret_cast<float*>(dyn),
                                                                            j0, n, acc);
    if (p.from_scores)  // the compaction reads them back
#pragma unroll
        for (int i = 0; i < PER; ++i)
            if (i < nvalid) pooled[j0 + jl + i] = acc[i];
    uint32_t key[PER], bins[PER];
#pragma unroll
    for (int i = 0; i < PER; ++i) {
        key[i] = rank_key(acc[i]);
        bins[i] = key[i] >> kHistShift;
    }
    // first-digit counts of the chunk
    for (int b = tid; b < kHistBins; b += kSelThreads) sh.hist[b] = 0;
    __syncthreads();
    add_runs<PER>(sh.hist, bins, nvalid);
    __syncthreads();
    // group starts, highest digit first; the unit's counts
    const size_t slot = static_cast<size_t>(unit) * p.max_chunks + c;
    int* cs = p.chunk_start + slot * kHistBins;
    int* gh = p.hist + static_cast<size_t>(unit) * kHistBins;
    {
        constexpr int BPT = kHistBins / kSelThreads;
        const int base = (kSelThreads - 1 - tid) * BPT;
        int h[BPT], local = 0;
#pragma unroll
        for (int q = BPT - 1; q >= 0; --q) {
            h[q] = sh.hist[base + q];
            local += h[q];
        }
        int tot;
        int start = block_excl_scan<kSelThreads>(local, sh.scratch, &tot);
#pragma unroll
        for (int q = BPT - 1; q >= 0; --q) {
            sh.fill[base + q] = start;
            cs[base + q] = start;
            if (h[q]) atomicAdd(gh + base + q, h[q]);
            start += h[q];
        }
    }
    __syncthreads();
    // the chunk's (key, position) pairs grouped by first digit; a run of equal digits takes
    // consecutive slots
    uint2* bk = p.buckets + slot * kChunk;
    {
        int at = 0;
#pragma unroll
        for (int i = 0; i < PER; ++i) {
            if (i < nvalid) {
                if (i == 0 || bins[i] != bins[i - 1]) {
                    int len = 1;
                    bool run = true;
#pragma unroll
                    for (int q = i + 1; q < PER; ++q) {
                        run = run && q < nvalid && bins[q] == bins[i];
                        len += run ? 1 : 0;
                    }
                    at = atomicAdd(&sh.fill[bins[i]], len);
                } else {
                    ++at;
                }
                bk[at] = make_uint2(key[i], static_cast<uint32_t>(j0 + jl + i));
            }
        }
    }
    // The last chunk block of the unit to get here computes the unit's threshold.  The
    // barrier orders the block's stores before thread 0's release; its acquire, and the
    // barrier after it, order the other blocks' stores before this block's reads.
    __syncthreads();
    if (tid == 0) sh.last = atomic_add_acq_rel(p.arrivals + unit, 1) == nch - 1;
    __syncthreads();
    if (!sh.last) return;
    unit_threshold(p, u, unit, nch, sh, dyn);
}

__global__ void __launch_bounds__(kSelThreads) compact_kernel(const __grid_constant__ SelectParams p) {
    extern __shared__ int list[];  // [kChunk] the chunk's kept positions, in order
    __shared__ int wbase[kSelWarps + 1];
    const int unit = blockIdx.x, c = blockIdx.y, tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    if (unit == 0 && c == 0 && tid == 0 && seqlens_hash(p.cu_seqlens, p.S) != p.cu_hash)
        record_error(p.status, kDevBadSeqlens, 220);
    UnitGeo u;
    if (!unit_geo(p, unit, u)) return;
    if (u.L <= kUnitLen) return;  // select_unit_kernel took it
    if (u.g == 0 && c == 0 && tid == 0) {
        p.cu_keep[u.s + 1] = u.keep_off + u.n_keep;
        if (u.s == 0) p.cu_keep[0] = 0;
    }
    const int j0 = c * kChunk;
    if (u.L <= p.budget) {  // kept whole
        const int m = max(0, min(u.L, j0 + kChunk) - j0);
        for (int e = tid; e < m; e += kSelThreads) list[e] = j0 + e;
        __syncthreads();
        emit_kept(p, u, list, m, j0, u.g * (p.Hkv / p.n_vec), (u.g + 1) * (p.Hkv / p.n_vec));
        return;
    }
    const int P = u.P, k = u.k;
    if (c == 0) {  // the window closes the list
        for (int i = tid; i < p.w; i += kSelThreads) list[i] = P + i;
        __syncthreads();
        emit_kept(p, u, list, p.w, k, u.g * (p.Hkv / p.n_vec), (u.g + 1) * (p.Hkv / p.n_vec));
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
        for (int x = 0; x < kSelWarps; ++x) {
            const int t = wbase[x];
            wbase[x] = a;
            a += t;
        }
        wbase[kSelWarps] = a;
    }
    __syncthreads();
    const int tot = wbase[kSelWarps];
    if (base < 0 || base + tot > k) {
        if (tid == 0) record_error(p.status, kDevBadIndex, 320 + unit);
        return;
    }
    int r = wbase[warp];
    const unsigned lt = (1u << lane) - 1u;
#pragma unroll
    for (int q = 0; q < kIt; ++q) {
        if ((bal[q] >> lane) & 1u) list[r + __popc(bal[q] & lt)] = js + q * 32;
        r += __popc(bal[q]);
    }
    __syncthreads();
    emit_kept(p, u, list, tot, base, u.g * (p.Hkv / p.n_vec), (u.g + 1) * (p.Hkv / p.n_vec));
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

// ------------------------------------------------------------------ TMA stage
// A stage row of one score row for one chunk, loaded by TMA from the score buffer viewed as
// 16-float lines (64 bytes): kLsTmaBoxes boxes of kScoreMapBoxLines lines from the line holding
// position base-4 on, so element e of the row sits at position base-4-d+e, d = the offset of
// position base-4 in its line.  The TMA writes each 64-byte line with the 64-byte swizzle: the
// 16-byte chunk bits 4-5 of a byte offset XOR its bits 7-8 (rows 1024-byte aligned).  For the
// pooling's reads of 16 elements per thread that places the 16-byte reads of every
// quarter-warp in distinct bank groups.
constexpr int kLsTmaBoxes = 3;
constexpr int kLsTmaRow = kLsTmaBoxes * kScoreMapBoxLines * 16;   // floats per stage row
static_assert(kLsTmaRow >= 15 + 8192 + 8 + 3, "a chunk, its halo, the line offset and a shifted read fit a stage row");
static_assert((kLsTmaRow * 4) % 1024 == 0 && (kScoreMapBoxLines * 64) % 1024 == 0, "1024-byte aligned boxes");
__device__ __forceinline__ int sw64(int byte) { return byte ^ (((byte >> 7) & 3) << 4); }

__device__ __forceinline__ float fmax3(float a, float b, float c) {
    float d;
    asm("max.f32 %0, %1, %2, %3;" : "=f"(d) : "f"(a), "f"(b), "f"(c));
    return d;
}
// Asks L2 to fetch bytes [p, p + n) (16-byte aligned, n a multiple of 16): a hint that moves
// nothing into the SM, so that a later copy of the same bytes finds them in L2.
__device__ __forceinline__ void prefetch_l2(const void* p, uint32_t n) {
    asm volatile("cp.async.bulk.prefetch.L2.global [%0], %1;" ::"l"(p), "r"(n) : "memory");
}

// prefetch_l2 of positions [a, b) of a score row, clamped to [0, P) and trimmed to whole
// 16-byte groups.
__device__ __forceinline__ void prefetch_row_l2(const float* row, int a, int b, int P) {
    a = max(a, 0);
    b = min(b, P);
    if (b <= a) return;
    const uintptr_t s = (reinterpret_cast<uintptr_t>(row + a) + 15) & ~static_cast<uintptr_t>(15);
    const uintptr_t e = reinterpret_cast<uintptr_t>(row + b) & ~static_cast<uintptr_t>(15);
    if (e > s) prefetch_l2(reinterpret_cast<const void*>(s), static_cast<uint32_t>(e - s));
}

// Issues, from one thread, the TMA loads that stage score rows ra .. ra+nr-1 of the chunk at
// `base` (row i at st + i*words), completion on `bar`.  Earlier generic-proxy writes to the
// stage (the previous unit's kept list) are ordered before the loads by the proxy fence.
__device__ __forceinline__ void stage_rows_tma(float* st, int words, const CUtensorMap* map, uint64_t* bar,
                                               size_t T, int t0, int ra, int nr, int base) {
    fence_proxy_async_smem();
    mbar_arrive_expect_tx(bar, static_cast<uint32_t>(nr * kLsTmaRow * 4));
    for (int i = 0; i < nr; ++i) {
        const long long f = static_cast<long long>(ra + i) * static_cast<long long>(T) + t0 + base - 4;
        const int line = f >= 0 ? static_cast<int>(f >> 4) : -1;  // f >= -4; line -1 reads zeros
        for (int b = 0; b < kLsTmaBoxes; ++b)
            tma_load_2d(st + i * words + b * kScoreMapBoxLines * 16, map, bar, 0, line + b * kScoreMapBoxLines);
    }
}

// The line offset d of row ra+i's chunk at `base` in its stage row (stage_rows_tma).
__device__ __forceinline__ int stage_offset(size_t T, int t0, int r, int base) {
    const long long f = static_cast<long long>(r) * static_cast<long long>(T) + t0 + base - 4;
    return f >= 0 ? static_cast<int>(f & 15) : static_cast<int>(f + 16);
}

// Pools the PER = 16 outputs of thread t (positions base+16t .. base+16t+15) from one stage
// row: its 24 elements d+16t .. d+16t+23 (positions base-4+16t ..), d = 4a + SHIFT, in six
// 16-byte reads from element 4a+16t on (seven when SHIFT > 0), those outside [0, P) taken as
// zero; output i covers elements 16t+i+4-HALF .. 16t+i+4+HALF.  The same arithmetic, in the
// same order, as pool_window.
template <int HALF, int SHIFT, int PER>
__device__ __forceinline__ void pool_window_tma(const float* row, int d, int t, int nvalid, bool is_max,
                                                float kf, int pos0, int P, float (&acc)[PER]) {
    static_assert(PER == 16 && HALF >= 0 && HALF <= 4 && SHIFT >= 0 && SHIFT < 4, "window");
    constexpr int kReads = SHIFT > 0 ? 7 : 6;
    float r[4 * kReads];
    const char* rb = reinterpret_cast<const char*>(row);
    const int e0 = (d & ~3) + 16 * t;
#pragma unroll
    for (int q = 0; q < kReads; ++q) {
        const float4 x = *reinterpret_cast<const float4*>(rb + sw64(4 * (e0 + 4 * q)));
        r[4 * q] = x.x;
        r[4 * q + 1] = x.y;
        r[4 * q + 2] = x.z;
        r[4 * q + 3] = x.w;
    }
    float w[24];
#pragma unroll
    for (int j = 0; j < 24; ++j) w[j] = r[SHIFT + j];
    const int p0 = pos0 + 16 * t;  // position of w[0]
    if (p0 < 0 || p0 + 24 > P) {
#pragma unroll
        for (int j = 0; j < 24; ++j)
            if (p0 + j < 0 || p0 + j >= P) w[j] = 0.f;
    }
    if (is_max) {
        // maxima of three neighbours, shared by the windows that contain them (a maximum is
        // exact in any order)
        float m3[22];
#pragma unroll
        for (int j = 0; j < 22; ++j) m3[j] = fmax3(w[j], w[j + 1], w[j + 2]);
#pragma unroll
        for (int i = 0; i < PER; ++i) {
            if (i < nvalid) {
                constexpr int W = 2 * HALF + 1;
                const int s0 = i + 4 - HALF;
                float m;
                if (W == 1) m = w[s0];
                else if (W == 3) m = m3[s0];
                else if (W == 5) m = fmax3(m3[s0], w[s0 + 3], w[s0 + 4]);
                else if (W == 7) m = fmax3(m3[s0], m3[s0 + 3], w[s0 + 6]);
                else m = fmax3(m3[s0], m3[s0 + 3], m3[s0 + 6]);
                acc[i] += m;
            }
        }
    } else {
#pragma unroll
        for (int i = 0; i < PER; ++i) {
            if (i < nvalid) {
                float m = w[i + 4 - HALF];
#pragma unroll
                for (int dd = 1; dd <= 2 * HALF; ++dd) m += w[i + 4 - HALF + dd];
                acc[i] += m / kf;  // IEEE division, as in pool_kernel
            }
        }
    }
}

template <int HALF, int PER>
__device__ __forceinline__ void pool_shift_tma(const float* row, int d, int t, int nvalid, bool is_max,
                                               float kf, int pos0, int P, float (&acc)[PER]) {
    const int shift = d & 3;  // the same for every thread of the block
    if (shift == 0) pool_window_tma<HALF, 0, PER>(row, d, t, nvalid, is_max, kf, pos0, P, acc);
    else if (shift == 1) pool_window_tma<HALF, 1, PER>(row, d, t, nvalid, is_max, kf, pos0, P, acc);
    else if (shift == 2) pool_window_tma<HALF, 2, PER>(row, d, t, nvalid, is_max, kf, pos0, P, acc);
    else pool_window_tma<HALF, 3, PER>(row, d, t, nvalid, is_max, kf, pos0, P, acc);
}

template <int PER>
__device__ __forceinline__ void pool_any_tma(const float* row, int d, int t, int nvalid, int half, bool is_max,
                                             float kf, int pos0, int P, float (&acc)[PER]) {
    if (nvalid <= 0) return;
    if (half == 3) pool_shift_tma<3, PER>(row, d, t, nvalid, is_max, kf, pos0, P, acc);
    else if (half == 2) pool_shift_tma<2, PER>(row, d, t, nvalid, is_max, kf, pos0, P, acc);
    else if (half == 1) pool_shift_tma<1, PER>(row, d, t, nvalid, is_max, kf, pos0, P, acc);
    else if (half == 0) pool_shift_tma<0, PER>(row, d, t, nvalid, is_max, kf, pos0, P, acc);
    else pool_shift_tma<4, PER>(row, d, t, nvalid, is_max, kf, pos0, P, acc);
}

// ------------------------------------------------------------------ many layers at once
// Selection of every (layer, sequence, selection) unit of a multi-layer call in one launch:
// the CTAs take units from a global counter, and one CTA does a unit whole, streaming over its
// candidate positions in chunks of kLsChunk (so that no length is too long and little sits in
// shared memory):
//  (A) pools the chunk (the next chunk's score rows copied in meanwhile) and appends the keys
//      that can still be kept, with their positions, to the unit's candidate list in a scratch
//      row: the first digits of the order-preserving keys are counted until the chunks so far
//      hold k keys; the first digit of their k-th largest then bounds the unit's k-th largest
//      from below, and later keys under it are not listed (the digits of later candidates are
//      counted from the list before (B));
//  (B) finds the k-th largest key from the counts (the first digit) and two more digits (11 and
//      10 bits) counted over the candidates with the digits so far: gathered into shared memory
//      when at most kLsCand share the first digit, else read from the list; the tie cutoff
//      among keys equal to the threshold is their rank by position, in shared memory when at
//      most kLsTies were gathered, else by a scan of the list (which is in position order);
//  (C) writes the kept candidates' positions in order (a block scan per kLsChunk of the list)
//      with their K/V rows, and appends the window.
// The same keys, ties and order as select_unit_kernel and the chunked kernels.
constexpr int kLsThreads = 512;
constexpr int kLsPer = 16;
constexpr int kLsChunk = kLsThreads * kLsPer;                    // 8192 positions
constexpr int kLsStageFloats = kLsChunk + 2 * kMaxHalo;
constexpr int kLsStageLoads = (kLsStageFloats + kLsThreads - 1) / kLsThreads;
// four score rows at once in the padded layout, or two buffers of two TMA stage rows (plus the
// slack that aligns them to 1024 bytes)
constexpr int kLsWords = 4 * stage_words(kLsStageFloats) > 4 * kLsTmaRow + 256 ? 4 * stage_words(kLsStageFloats)
                                                                               : 4 * kLsTmaRow + 256;
constexpr int kLsList = kLsWords;                                // kept positions gathered at once
static_assert(kLsList >= kLsChunk, "a chunk's kept positions fit the list");
constexpr int kLsSmem = kLsWords * 4;
constexpr int kLsAhead = 2;     // score-row chunks asked into L2 ahead of the one being copied in
constexpr int kLsCand = 2048;   // keys sharing the k-th key's first digit gathered in shared memory
constexpr int kLsTies = 256;    // keys equal to the k-th key ranked by position in shared memory
constexpr int kSelMaxLayers = 32;

struct SelectLayersParams {
    CUtensorMap score_map[kSelMaxLayers];  // each layer's scores as 16-float lines (map_mask)
    uint32_t map_mask;                     // bit i: score_map[i] is set
    SelectParams layer[kSelMaxLayers];
    uint2* cands[kSelMaxLayers];     // per layer [n_vec, key_stride]: (key, position) candidates
    int* next_unit;                  // work counter, zero at launch
    int n_layers, units_per_layer;   // units_per_layer = S * n_vec
    int key_stride;                  // select_key_stride(T, S)
};

__global__ void __launch_bounds__(kLsThreads, 1) select_layers_kernel(const __grid_constant__ SelectLayersParams P) {
    extern __shared__ __align__(16) float st[];  // pooling stage; the kept list of a chunk
    __shared__ int hist[kHistBins];
    __shared__ int scratch[33];
    __shared__ int wsum[2][kLsThreads / 32];  // the one-barrier scans' warp sums, alternating
    __shared__ int s_digit, s_above, s_cut, s_cnt, s_unit;
    __shared__ uint32_t s_thr;
    __shared__ uint2 cand[kLsCand];
    __shared__ uint64_t tbar[2];  // TMA stage buffers: the loads of a chunk complete
    __shared__ int s_abort;
    constexpr int NT = kLsThreads, PER = kLsPer;
    const int tid = threadIdx.x;
    float* const sta = reinterpret_cast<float*>((reinterpret_cast<uintptr_t>(st) + 1023) & ~static_cast<uintptr_t>(1023));
    uint32_t tph = 0;  // bit b: parity of the next completion of tbar[b]
    if (tid == 0) {
        mbar_init(&tbar[0], 1);
        mbar_init(&tbar[1], 1);
        s_abort = 0;
        fence_mbar_init();
    }
    if (blockIdx.x == 0 && tid == 0) {
        const SelectParams& p0 = P.layer[0];
        if (seqlens_hash(p0.cu_seqlens, p0.S) != p0.cu_hash) record_error(p0.status, kDevBadSeqlens, 240);
    }
    const int n_units = P.n_layers * P.units_per_layer;
    for (;;) {
        if (tid == 0) s_unit = atomicAdd(P.next_unit, 1);
        fence_proxy_async_smem();  // this thread's writes to the stage before the unit's TMA loads
        __syncthreads();
        const int gu = s_unit;
        __syncthreads();
        if (gu >= n_units) break;
        const int li = gu / P.units_per_layer, lu = gu % P.units_per_layer;
        const SelectParams& p = P.layer[li];
        // One selection per layer (n_vec = 1) is made by H_kv units, each writing the positions
        // and copying the rows of one KV head, so that the row copies spread over CTAs; every
        // copy of the selection is the same (the same inputs and steps).
        const int copies = p.n_vec == 1 ? p.Hkv : 1, cu = lu % copies, unit = lu / copies;
        UnitGeo u;
        if (!unit_geo(p, unit, u)) continue;
        const int kv0 = p.n_vec == p.Hkv ? u.g : cu, kv1 = kv0 + 1;
        if (u.g == 0 && cu == 0 && tid == 0) {
            p.cu_keep[u.s + 1] = u.keep_off + u.n_keep;
            if (u.s == 0) p.cu_keep[0] = 0;
        }
        float* pooled = p.write_pooled && cu == 0 ? p.pooled + static_cast<size_t>(u.g) * p.T + u.t0 : nullptr;
        int* list = reinterpret_cast<int*>(st);
        if (u.L <= p.budget) {  // kept whole; its pooled scores read as 0
            for (int e0 = 0; e0 < u.L; e0 += kLsChunk) {
                const int m = min(kLsChunk, u.L - e0);
                for (int e = tid; e < m; e += NT) {
                    list[e] = e0 + e;
                    if (pooled) pooled[e0 + e] = 0.f;
                }
                __syncthreads();
                emit_kept(p, u, list, m, e0, kv0, kv1);
                __syncthreads();
            }
            continue;
        }
        const int Pn = u.P, k = u.k;
        // the unit's candidate list of (key, position) pairs: sequence s's segment of the
        // scratch row starts at its first token rounded up to a multiple of 4, plus 4 s, so that
        // every segment is 32-byte aligned and holds the sequence's P candidates at most
        uint2* cands = P.cands[li] + static_cast<size_t>(u.g * copies + cu) * P.key_stride + ((u.t0 + 3) & ~3) + 4 * u.s;
        int n_cand = 0;
        if (pooled)  // window positions are not candidates
            for (int j = Pn + tid; j < u.L; j += NT) pooled[j] = 0.f;
        // (A) pooled scores, keys and first-digit counts, chunk by chunk
        for (int b = tid; b < kHistBins; b += NT) hist[b] = 0;
        // With the heads pooled one by one and two chunks' rows fitting the stage, the next
        // chunk's rows are copied in while this chunk is pooled (two buffers of nr rows).
        const int half = p.pool_kernel >> 1;
        const int r0 = p.group_first[u.g], nr = p.group_first[u.g + 1] - r0;
        // TMA staging when the pooling window fits a thread's 24 staged elements and the unit's
        // rows fit the stage, in two buffers (the next chunk loaded while this one is pooled)
        // or else one; otherwise 4-byte copies in the padded layout
        const bool tma = ((P.map_mask >> li) & 1u) && p.from_scores && p.head_order == 0 && half <= 4 &&
                         nr * kLsTmaRow + 256 <= kLsWords;
        const int nb = tma && 2 * nr * kLsTmaRow + 256 > kLsWords ? 1 : 2;  // stage buffers
        const int words = tma ? kLsTmaRow : stage_words(kLsChunk + 2 * half);
        const bool piped = tma || (p.from_scores && p.head_order == 0 && 2 * nr * words + PER <= kLsWords);
        float* const stg = tma ? sta : st;
        if (tma) {
            if (tid == 0) stage_rows_tma(stg, words, &P.score_map[li], &tbar[0], p.T, u.t0, r0, nr, 0);
        } else if (piped)
            stage_rows_issue<NT, kLsStageLoads>(st, words, p.scores, p.T, u.t0, r0, nr, 0, half,
                                                min(kLsChunk, Pn), u.P);
        // The chunks after the next are asked into L2 kLsAhead chunks ahead of their copy, so
        // that the copies overlapped with pooling find them there.
        const float* srow = p.scores + static_cast<size_t>(r0 + tid) * p.T + u.t0;
        if (piped && tid < nr)
            for (int d = 1; d <= kLsAhead; ++d)
                prefetch_row_l2(srow, d * kLsChunk - 4, (d + 1) * kLsChunk + 4, Pn);
        __syncthreads();
        uint32_t lo = 0;  // the lowest first digit counted (see below)
        int n_hist = -1;  // candidates from n_hist on are not counted in hist (see below)
        for (int base = 0, c = 0; base < Pn; base += kLsChunk, ++c) {
            const int n = min(kLsChunk, Pn - base);
            const int jb = tid * PER, nvalid = n - jb;
            float acc[PER];
            if (piped) {
                const int bi = nb == 2 ? (c & 1) : 0;
                const float* cur = stg + bi * nr * words;
                const bool more = base + kLsChunk < Pn;
                // one buffer: chunk c > 0 is loaded now, its buffer freed by the last chunk's barrier
                if (nb == 1 && c > 0 && tid == 0)
                    stage_rows_tma(stg, words, &P.score_map[li], &tbar[0], p.T, u.t0, r0, nr, base);
                if (more && nb == 2) {
                    float* nxt_st = stg + ((c + 1) & 1) * nr * words;
                    const int nn = min(kLsChunk, Pn - base - kLsChunk);
                    if (tma) {
                        if (tid == 0)
                            stage_rows_tma(nxt_st, words, &P.score_map[li], &tbar[(c + 1) & 1], p.T, u.t0, r0, nr,
                                           base + kLsChunk);
                    } else {
                        stage_rows_issue<NT, kLsStageLoads>(nxt_st, words, p.scores, p.T, u.t0, r0, nr,
                                                            base + kLsChunk, half, nn, u.P);
                    }
                    if (!tma) cp_async_wait_group<1>();
                } else if (!tma) {
                    cp_async_wait_group<0>();
                }
                if (more && tid < nr) {
                    const int a = base + (1 + kLsAhead) * kLsChunk;
                    prefetch_row_l2(srow, a - 4, a + kLsChunk + 4, Pn);
                }
                if (tma) {  // this chunk's loads have landed (a bounded wait)
                    const int b = bi;
                    const bool ok = mbar_wait(&tbar[b], (tph >> b) & 1u, &s_abort);
                    tph ^= 1u << b;
                    if (__syncthreads_or(ok ? 0 : 1)) {
                        // give up: report, let the loads still in flight land, leave
                        if (tid == 0) {
                            record_error(p.status, kDevTimeout, 250);
                            volatile int never = 0;
                            mbar_wait(&tbar[b], ((tph >> b) & 1u) ^ 1u, &never);
                            if (more && nb == 2) mbar_wait(&tbar[b ^ 1], (tph >> (b ^ 1)) & 1u, &never);
                        }
                        return;
                    }
                } else {
                    __syncthreads();
                }
#pragma unroll
                for (int i = 0; i < PER; ++i) acc[i] = 0.f;
                for (int i = 0; i < nr; ++i) {
                    if (tma)
                        pool_any_tma<PER>(cur + i * words, stage_offset(p.T, u.t0, r0 + i, base), tid, nvalid, half,
                                          p.pool_type == 0, static_cast<float>(p.pool_kernel), base - 4, Pn, acc);
                    else
                        pool_any<PER>(cur + i * words, jb, nvalid, half, p.pool_type == 0,
                                      static_cast<float>(p.pool_kernel), acc);
                }
            } else {
                pooled_values<NT, PER, kLsStageLoads, kLsWords>(p, u, st, base, n, acc);
            }
            uint32_t key[PER];  // first digit: key >> kHistShift
#pragma unroll
            for (int i = 0; i < PER; ++i) key[i] = rank_key(acc[i]);
            if (pooled) {  // 16-byte stores where the row is 16-byte aligned
                if (nvalid >= PER && (reinterpret_cast<uintptr_t>(pooled) & 15u) == 0) {
#pragma unroll
                    for (int q = 0; q < PER / 4; ++q)
                        reinterpret_cast<float4*>(pooled + base + jb)[q] =
                            make_float4(acc[4 * q], acc[4 * q + 1], acc[4 * q + 2], acc[4 * q + 3]);
                } else {
#pragma unroll
                    for (int i = 0; i < PER; ++i)
                        if (i < nvalid) pooled[base + jb + i] = acc[i];
                }
            }
            // Once the bound is set, a chunk is not counted here: (B) adds the first digits of
            // its candidates (its only keys that can be kept) from the list instead.
            if (lo == 0) add_runs<PER, kHistShift>(hist, key, nvalid, lo);
            else if (n_hist < 0) n_hist = n_cand;
            if (lo == 0 && k > 0) {
                // The k-th largest key of the chunks so far bounds the unit's k-th largest from
                // below: in later chunks only keys whose first digit is at or above its digit can
                // be kept, and the counts at or above it, which the threshold search reads, stay
                // exact when only those keys are counted.
                __syncthreads();
                find_digit<NT>(hist, k, scratch, &s_digit, &s_above);
                lo = static_cast<uint32_t>(s_digit);  // 0 while fewer than k keys are counted
            }
            if (k > 0) {  // the candidates, in position order: keys whose first digit is >= lo
                int cnt = 0;
#pragma unroll
                for (int i = 0; i < PER; ++i) cnt += (i < nvalid && (key[i] >> kHistShift) >= lo) ? 1 : 0;
                int tot;
                int off = n_cand + block_excl_scan1<NT>(cnt, wsum[c & 1], &tot);
#pragma unroll
                for (int i = 0; i < PER; ++i)
                    if (i < nvalid && (key[i] >> kHistShift) >= lo)
                        cands[off++] = make_uint2(key[i], static_cast<uint32_t>(base + jb + i));
                n_cand += tot;
            }
            if (piped) __syncthreads();  // every thread is done with this chunk's buffer
        }
        __syncthreads();  // the candidates and counts are complete (same block)
        // (B) the k-th largest key thr, and the last position cut of a kept key equal to it
        // (k = 0 keeps only the window: no key is above 0xffffffff, no position at or below -1)
        uint32_t thr = 0xFFFFFFFFu;
        int pos_cut = -1;
        if (k > 0) {
            if (tid == 0) s_cut = INT_MAX;
            if (n_hist >= 0) {  // the first digits of the candidates of the chunks not counted in (A)
                for (int c = n_hist + tid; c < n_cand; c += NT) atomicAdd(&hist[__ldcg(cands + c).x >> kHistShift], 1);
                __syncthreads();
            }
            find_digit<NT>(hist, k, scratch, &s_digit, &s_above);
            const uint32_t d1 = static_cast<uint32_t>(s_digit);
            int r = k - s_above, n_eq = hist[d1];
            const int n_first = n_eq;
            __syncthreads();
            // The candidates with the k-th key's first digit: gathered into shared memory when
            // there are at most kLsCand of them (the usual case), else read from the list.
            const bool in_smem = n_eq <= kLsCand;
            if (in_smem) {
                if (tid == 0) s_cnt = 0;
                __syncthreads();
                for (int c = tid; c < n_cand; c += NT) {
                    const uint2 x = __ldcg(cands + c);
                    if ((x.x >> kHistShift) == d1) {
                        const int i = atomicAdd(&s_cnt, 1);
                        if (i < kLsCand) cand[i] = x;
                    }
                }
                __syncthreads();
            }
            // Two more digits (11 and 10 bits) of the k-th key, by counts of the keys that share
            // the digits so far.
            uint32_t prefix = d1 << kHistShift, mask = 0x7FFu << kHistShift;
#pragma unroll 1
            for (int level = 0; level < 2; ++level) {
                const int shift = level == 0 ? 10 : 0;
                const uint32_t dmask = level == 0 ? 0x7FFu : 0x3FFu;
                for (int b = tid; b < kHistBins; b += NT) hist[b] = 0;
                __syncthreads();
                if (in_smem) {
                    for (int c = tid; c < n_first; c += NT) {
                        const uint32_t kk = cand[c].x;
                        if ((kk & mask) == prefix) atomicAdd(&hist[(kk >> shift) & dmask], 1);
                    }
                } else {
                    for (int c = tid; c < n_cand; c += NT) {
                        const uint32_t kk = __ldcg(cands + c).x;
                        if ((kk & mask) == prefix) atomicAdd(&hist[(kk >> shift) & dmask], 1);
                    }
                }
                __syncthreads();
                find_digit<NT>(hist, r, scratch, &s_digit, &s_above);
                prefix |= static_cast<uint32_t>(s_digit) << shift;
                mask |= dmask << shift;
                r -= s_above;
                n_eq = hist[s_digit];  // now: the keys equal to the k-th key
                __syncthreads();
            }
            thr = prefix;
            const int need_eq = r;  // keys equal to thr that are kept: the lowest positions
            pos_cut = INT_MAX;
            if (need_eq < n_eq) {
                if (in_smem && n_eq <= kLsTies) {
                    // the candidates equal to thr, ranked by position in shared memory (the
                    // counts are no longer needed: their array holds the positions)
                    int* eq = hist;
                    if (tid == 0) s_cnt = 0;
                    __syncthreads();
                    for (int c = tid; c < n_first; c += NT) {
                        const uint2 x = cand[c];
                        if (x.x == thr) eq[atomicAdd(&s_cnt, 1)] = static_cast<int>(x.y);
                    }
                    __syncthreads();
                    for (int i = tid; i < n_eq; i += NT) {
                        const int me = eq[i];
                        int ahead = 0;
                        for (int q = 0; q < n_eq; ++q) ahead += eq[q] < me ? 1 : 0;
                        if (ahead == need_eq - 1) s_cut = me;
                    }
                    __syncthreads();
                    pos_cut = s_cut;
                } else {
                    // a scan of the list, which is in position order
                    int seen = 0;  // keys equal to thr in the chunks before
                    for (int b0 = 0; b0 < n_cand && seen < need_eq; b0 += kLsChunk) {
                        const int jb = tid * PER, nvalid = min(kLsChunk, n_cand - b0) - jb;
                        int ne = 0;
#pragma unroll
                        for (int i = 0; i < PER; ++i) ne += (i < nvalid && __ldcg(cands + b0 + jb + i).x == thr) ? 1 : 0;
                        int tot;
                        const int before = seen + block_excl_scan<NT>(ne, scratch, &tot);
                        if (before < need_eq && before + ne >= need_eq) {
                            int c = before;
#pragma unroll
                            for (int i = 0; i < PER; ++i) {
                                if (i < nvalid) {
                                    const uint2 x = __ldcg(cands + b0 + jb + i);
                                    if (x.x == thr && ++c == need_eq) s_cut = static_cast<int>(x.y);
                                }
                            }
                        }
                        seen += tot;
                    }
                    __syncthreads();
                    pos_cut = s_cut;
                }
            }
        }
        // (C) the kept positions in order: the candidates above the threshold, or equal to it
        // and at or before the tie cutoff, a block scan per kLsChunk of the list; gathered in
        // the stage (free now) and written out with their K/V rows when it is full and at the
        // end, so that the rows' copies share one round trip; then the window
        int written = 0, lbase = 0, lcount = 0;  // list[0..lcount) are output rows lbase..
        for (int b0 = 0; b0 < n_cand && k > 0; b0 += kLsChunk) {
            const int jb = tid * PER, nvalid = min(kLsChunk, n_cand - b0) - jb;
            uint32_t taken = 0;
            int cnt = 0, pos[PER];
#pragma unroll
            for (int q = 0; q < PER / 2; ++q) {
                // 16-byte loads: the list is 32-byte aligned, b0 + jb a multiple of 16
                uint4 x2 = make_uint4(0u, 0u, 0u, 0u);
                if (2 * q < nvalid) {
                    if (2 * q + 1 < nvalid) {
                        x2 = __ldcg(reinterpret_cast<const uint4*>(cands + b0 + jb) + q);
                    } else {
                        const uint2 x = __ldcg(cands + b0 + jb + 2 * q);
                        x2.x = x.x;
                        x2.y = x.y;
                    }
                }
                const uint32_t kx[2] = {x2.x, x2.z};
                const int px[2] = {static_cast<int>(x2.y), static_cast<int>(x2.w)};
#pragma unroll
                for (int e = 0; e < 2; ++e) {
                    const int i = 2 * q + e;
                    pos[i] = px[e];
                    if (i < nvalid && (kx[e] > thr || (kx[e] == thr && px[e] <= pos_cut))) {
                        taken |= 1u << i;
                        ++cnt;
                    }
                }
            }
            int tot;
            int rk = block_excl_scan1<NT>(cnt, wsum[(b0 / kLsChunk) & 1], &tot);
            if (written + tot > k) break;  // checked below
            if (lcount + tot > kLsList) {  // block-uniform: write out the list first
                emit_kept(p, u, list, lcount, lbase, kv0, kv1);
                lbase += lcount;
                lcount = 0;
                __syncthreads();
            }
            rk += lcount;
#pragma unroll
            for (int i = 0; i < PER; ++i) {
                if ((taken >> i) & 1u) {
                    list[rk] = pos[i];
                    ++rk;
                }
            }
            lcount += tot;
            written += tot;
        }
        if (written != k) {
            if (tid == 0) record_error(p.status, kDevBadIndex, 340 + unit);
            __syncthreads();  // every thread is done with the list before the next unit
            continue;
        }
        if (lcount + p.w > kLsList) {
            __syncthreads();
            emit_kept(p, u, list, lcount, lbase, kv0, kv1);
            lbase += lcount;
            lcount = 0;
            __syncthreads();
        }
        for (int i = tid; i < p.w; i += NT) list[lcount + i] = Pn + i;
        __syncthreads();
        emit_kept(p, u, list, lcount + p.w, lbase, kv0, kv1);
        __syncthreads();
    }
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
    for (int g = 0; g <= L.n_vec; ++g) p.group_first[g] = static_cast<int16_t>(L.group_first[g]);
    if (L.T == 0) return cudaSuccess;
    dim3 grid((L.T + 255) / 256, L.n_vec);
    NvtxRange range("pool_kernel");
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
    p.arrivals = L.arrivals;
    p.chunk_start = L.chunk_start;
    p.buckets = reinterpret_cast<uint2*>(L.buckets);
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
    p.n_vec = L.n_vec;
    p.pool_kernel = L.pool_kernel;
    p.pool_type = L.pool_type;
    p.head_order = L.head_order;
    p.from_scores = L.from_scores;
    p.write_pooled = L.write_pooled;
    p.cu_hash = L.cu_hash;
    for (int g = 0; g <= L.n_vec; ++g) p.group_first[g] = static_cast<int16_t>(L.group_first[g]);
    const int units = L.S * L.n_vec;
    if (units == 0 || L.max_chunks == 0) return cudaSuccess;
    if (L.max_chunks > 65535) return cudaErrorInvalidConfiguration;
    const size_t sel_smem = std::max(static_cast<size_t>(kSelStageSmem),
                                     sizeof(uint32_t) * 2 * kCandCap +
                                         sizeof(int) * (3 * static_cast<size_t>(L.max_chunks) + 1 + kTieCap));
    static size_t sel_smem_set = 0;
    static bool configured = false;
    cudaError_t e;
    if (!configured) {
        e = cudaFuncSetAttribute(compact_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, kCompactSmem);
        if (e != cudaSuccess) return e;
        e = cudaFuncSetAttribute(select_unit_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, kUnitSmem);
        if (e != cudaSuccess) return e;
        configured = true;
    }
    if (sel_smem > sel_smem_set) {
        e = cudaFuncSetAttribute(select_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                 static_cast<int>(sel_smem));
        if (e != cudaSuccess) return e;
        sel_smem_set = sel_smem;
    }
    if (L.min_len <= kUnitLen) {
        NvtxRange range("select_unit_kernel");
        select_unit_kernel<<<units * (L.Hkv / L.n_vec), kUnitThreads, kUnitSmem, stream>>>(p);
        if ((e = cudaGetLastError()) != cudaSuccess) return e;
    }
    if (L.max_len > kUnitLen) {
        NvtxRange range("select_kernel+compact_kernel");
        const dim3 grid(units, L.max_chunks);
        select_kernel<<<grid, kSelThreads, sel_smem, stream>>>(p);
        if ((e = cudaGetLastError()) != cudaSuccess) return e;
        compact_kernel<<<grid, kSelThreads, kCompactSmem, stream>>>(p);
        if ((e = cudaGetLastError()) != cudaSuccess) return e;
    }
    return cudaSuccess;
}

int select_chunks(int max_len) { return max(1, (max_len + kChunk - 1) / kChunk); }
size_t select_hist_ints() { return kHistBins; }
int select_chunk_positions() { return kChunk; }
int select_unit_len() { return kUnitLen; }

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
    NvtxRange range("gather_kernel");
    gather_kernel<<<static_cast<unsigned>((rows + 7) / 8), 256, 0, stream>>>(p);
    return cudaGetLastError();
}

// The selection of several layers in one launch (select_layers_kernel); Ls[i] as for
// launch_select with from_scores = 1, and keys[i] a [H_kv, select_key_stride(T, S)] scratch of
// 8-byte (key, position) slots per layer.  One launch per
// kSelMaxLayers layers; `next_unit` (kSelMaxLayers-aligned count of ints) is the work counter
// of each launch and is cleared first.
int select_key_stride(int T, int S) { return (T + 4 * S + 3) & ~3; }

cudaError_t launch_select_layers(const SelectLaunch* Ls, uint32_t* const* keys, int n_layers,
                                 int* next_unit, int grid, cudaStream_t stream) {
    static SelectLayersParams P;  // ~25 KB; calls are serialised by `mu`
    static std::mutex mu;
    static_assert(sizeof(SelectLayersParams) <= 32000, "kernel parameters");
    std::lock_guard<std::mutex> lock(mu);
    static bool configured = false;
    if (!configured) {
        const cudaError_t e = cudaFuncSetAttribute(select_layers_kernel,
                                                   cudaFuncAttributeMaxDynamicSharedMemorySize, kLsSmem);
        if (e != cudaSuccess) return e;
        configured = true;
    }
    for (int l0 = 0; l0 < n_layers; l0 += kSelMaxLayers) {
        const int nl = std::min(kSelMaxLayers, n_layers - l0);
        memset(&P, 0, sizeof P);
        // The layers with the largest budgets (the longest gathers) first: the CTAs take units
        // in order, so the last ones taken are the shortest.
        int order[kSelMaxLayers];
        for (int i = 0; i < nl; ++i) order[i] = l0 + i;
        std::stable_sort(order, order + nl, [&](int a, int b) { return Ls[a].budget > Ls[b].budget; });
        for (int i = 0; i < nl; ++i) {
            const SelectLaunch& L = Ls[order[i]];
            SelectParams& p = P.layer[i];
            p.scores = L.scores;
            p.pooled = L.pooled;
            p.idx = L.idx;
            p.cu_keep = L.cu_keep_dev;
            p.cu_seqlens = L.cu_seqlens_dev;
            p.status = L.status;
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
            p.n_vec = L.n_vec;
            p.pool_kernel = L.pool_kernel;
            p.pool_type = L.pool_type;
            p.head_order = L.head_order;
            p.from_scores = 1;
            p.write_pooled = L.write_pooled;
            p.cu_hash = L.cu_hash;
            for (int g = 0; g <= L.n_vec; ++g) p.group_first[g] = static_cast<int16_t>(L.group_first[g]);
            P.cands[i] = reinterpret_cast<uint2*>(keys[order[i]]);
            if (L.score_map) {
                P.score_map[i] = *L.score_map;
                P.map_mask |= 1u << i;
            }
        }
        P.n_layers = nl;
        P.units_per_layer = Ls[l0].S * Ls[l0].n_vec * (Ls[l0].n_vec == 1 ? Ls[l0].Hkv : 1);
        P.key_stride = select_key_stride(Ls[l0].T, Ls[l0].S);
        P.next_unit = next_unit;
        const int units = nl * P.units_per_layer;
        if (units == 0) continue;
        cudaError_t e = cudaMemsetAsync(next_unit, 0, sizeof(int), stream);
        if (e != cudaSuccess) return e;
        NvtxRange range("select_layers_kernel");
        select_layers_kernel<<<std::min(grid, units), kLsThreads, kLsSmem, stream>>>(P);
        if ((e = cudaGetLastError()) != cudaSuccess) return e;
    }
    return cudaSuccess;
}

}  // namespace ckv
