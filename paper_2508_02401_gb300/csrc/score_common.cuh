// Pieces shared by the two window-scoring kernels (score_kernel.cu, score_resident.cu): the
// launch parameters, the warp roles' common constants and the epilogue arithmetic.
#pragma once

#include "ckv_device.cuh"
#include "ckv_internal.h"

namespace ckv {

constexpr int kTileBytes = kTileKeys * kHeadDim * 2;  // 32 KiB
constexpr int kHalfBytes = kTileBytes / 2;            // 64 dims x 128 keys
// The running maximum of a column is only moved when a logit exceeds it by more than 2^60:
// the running sum then stays far below the fp32 range (at most keys * 2^60), and terms that
// are 2^-126 below the reference are negligible against the reference term itself.
constexpr float kLazyTau = 60.0f;
constexpr int kCols = 32;                             // columns per epilogue warpgroup
constexpr int kThreads = 512;
constexpr int kWarpA = 4, kWarpB = 12;                // first pass-1 / pass-2 warp

struct alignas(128) ScoreParams {
    CUtensorMap tmap_k;            // K as {128 (dim), H_kv, T}, box {64, 1, 128}, 128B swizzle
    CUtensorMap tmap_q;            // q_win as {128, H_q, S*w}, box {64, 1, W_PAD}, 128B swizzle
    const __nv_bfloat16* q_win;    // [S, w, H_q, 128] packed
    const int32_t* cu_seqlens;     // device [S+1] (checked against cu_hash)
    float2* partials;              // [n_items, N]: (max, sum) per window-row column
    int* counters;                 // [n_units] arrivals, zero at launch
    float* scores;                 // [n_sel, T]
    int* status;
    int S, T, Hq, w, n_rounds, n_items, n_units;
    uint32_t cu_hash;
    float sl2;                     // softmax scale * log2(e)
    long long wait_cycles;         // limit of a bounded wait (ckv_set_wait_limit_us)
    const float* lse;              // given lse of the window rows (natural log), [Hq][lse_stride]
    long long lse_stride;
    int16_t batch_group[kMaxBatches];   // KV head of each head batch
    int16_t batch_first[kMaxBatches];   // score row of the batch's first head
    int16_t batch_nheads[kMaxBatches];  // heads in the batch
    int16_t sel_heads[kMaxQHeads];      // query head of each score row
    ScoreItem items[kMaxScoreItems];    // [n_rounds * gridDim.x]
    ScoreUnit units[kMaxScoreUnits];
};

__device__ __forceinline__ float redux_max(float v) {
    float r;
    asm volatile("redux.sync.max.f32 %0, %1, 0xffffffff;" : "=f"(r) : "f"(v));
    return r;
}

__device__ __forceinline__ void red_release_add(int* p, int v) {
    asm volatile("red.release.gpu.global.add.s32 [%0], %1;" ::"l"(p), "r"(v) : "memory");
}

__device__ __forceinline__ float lg2_approx(float x) {
    float y;
    asm("lg2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
    return y;
}

// Packed fp32 pairs (sm_100+): one instruction for two lanes' worth of FMA / add, with the
// same IEEE rounding as the scalar forms.
__device__ __forceinline__ void fma2(float& d0, float& d1, float a0, float a1, float b0, float b1,
                                     float c0, float c1) {
    asm("{\n\t.reg .b64 a, b, c, d;\n\t"
        "mov.b64 a, {%2, %3};\n\tmov.b64 b, {%4, %5};\n\tmov.b64 c, {%6, %7};\n\t"
        "fma.rn.f32x2 d, a, b, c;\n\tmov.b64 {%0, %1}, d;\n\t}"
        : "=f"(d0), "=f"(d1)
        : "f"(a0), "f"(a1), "f"(b0), "f"(b1), "f"(c0), "f"(c1));
}
__device__ __forceinline__ void add2(float& d0, float& d1, float a0, float a1, float b0, float b1) {
    asm("{\n\t.reg .b64 a, b, d;\n\t"
        "mov.b64 a, {%2, %3};\n\tmov.b64 b, {%4, %5};\n\t"
        "add.rn.f32x2 d, a, b;\n\tmov.b64 {%0, %1}, d;\n\t}"
        : "=f"(d0), "=f"(d1)
        : "f"(a0), "f"(a1), "f"(b0), "f"(b1));
}
__device__ __forceinline__ void mul2(float& d0, float& d1, float a0, float a1, float b0, float b1) {
    asm("{\n\t.reg .b64 a, b, d;\n\t"
        "mov.b64 a, {%2, %3};\n\tmov.b64 b, {%4, %5};\n\t"
        "mul.rn.f32x2 d, a, b;\n\tmov.b64 {%0, %1}, d;\n\t}"
        : "=f"(d0), "=f"(d1)
        : "f"(a0), "f"(a1), "f"(b0), "f"(b1));
}
// Three-operand maximum (sm_100+).
__device__ __forceinline__ float max3(float a, float b, float c) {
    float d;
    asm("max.f32 %0, %1, %2, %3;" : "=f"(d) : "f"(a), "f"(b), "f"(c));
    return d;
}
__device__ __forceinline__ float max16(const float (&d)[16]) {
    const float a = max3(d[0], d[1], d[2]), b = max3(d[3], d[4], d[5]), c = max3(d[6], d[7], d[8]);
    const float e = max3(d[9], d[10], d[11]), f = max3(d[12], d[13], d[14]);
    return max3(max3(a, b, c), max3(e, f, d[15]), -INFINITY);
}
// Sum of 2C values held as C pairs (x[2i], x[2i+1]) by packed adds; the result is a pair.
template <int C2>
__device__ __forceinline__ void pair_tree(float* x) {
#pragma unroll
    for (int w = C2 / 2; w >= 2; w >>= 1)
#pragma unroll
        for (int i = 0; i < w; i += 2) add2(x[i], x[i + 1], x[i], x[i + 1], x[i + w], x[i + w + 1]);
}

__device__ __forceinline__ int ld_acquire(const int* p) {
    int v;
    asm volatile("ld.acquire.gpu.global.b32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
    return v;
}

template <int R>
__device__ __forceinline__ void setmaxnreg_inc() {
    asm volatile("setmaxnreg.inc.sync.aligned.u32 %0;" ::"n"(R));
}
template <int R>
__device__ __forceinline__ void setmaxnreg_dec() {
    asm volatile("setmaxnreg.dec.sync.aligned.u32 %0;" ::"n"(R));
}

// A barrier of one epilogue warpgroup on an mbarrier of kGroupArrivals arrivals, one per warp:
// each warp converges, its lane 0 arrives and waits (bounded, like every other wait of the
// kernel), and the warp converges again, which carries the ordering to the other lanes.
constexpr int kGroupArrivals = 4;
__device__ __forceinline__ bool group_sync(uint64_t* bar, uint32_t& phase, volatile int* abort,
                                           long long limit) {
    __syncwarp();
    int ok = 1;
    if ((threadIdx.x & 31) == 0) {
        mbar_arrive(bar);
        ok = mbar_wait(bar, phase, abort, limit) ? 1 : 0;
    }
    __syncwarp();
    ok = __shfl_sync(0xffffffffu, ok, 0);
    phase ^= 1;
    return ok != 0;
}

// Warp-wide sums of C per-lane columns (C = 8, 16 or 32) by recursive halving: at each level
// a lane keeps one half of its remaining columns and swaps the other half with its partner, so
// the C sums take C - 1 + log2(32 / C) shuffles instead of 5 C.  `m` (uniform across the warp)
// is carried along.  Afterwards lane l holds column l / (32 / C) in v[0] / m[0].
template <int C>
__device__ __forceinline__ void transpose_reduce(float (&v)[C], float (&m)[C], int lane) {
#pragma unroll
    for (int k = C / 2, bit = 16; k >= 1; k >>= 1, bit >>= 1) {
        const bool upper = (lane & bit) != 0;
#pragma unroll
        for (int i = 0; i < k; ++i) {
            const float send = upper ? v[i] : v[i + k];
            const float keep = upper ? v[i + k] : v[i];
            v[i] = keep + __shfl_xor_sync(0xffffffffu, send, bit);
            m[i] = upper ? m[i + k] : m[i];
        }
    }
#pragma unroll
    for (int bit = 16 / C; bit >= 1; bit >>= 1) v[0] += __shfl_xor_sync(0xffffffffu, v[0], bit);
}

// tcgen05.ld of 16 columns without the wait: the registers are not valid until tmem_ld_wait,
// and reg_fence then ties every later use to the wait.
__device__ __forceinline__ void tmem_ld16_nowait(uint32_t taddr, float (&v)[16]) {
    uint32_t r[16];
    asm volatile(
        "tcgen05.ld.sync.aligned.32x32b.x16.b32 "
        "{%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15}, [%16];"
        : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]),
          "=r"(r[7]), "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]),
          "=r"(r[13]), "=r"(r[14]), "=r"(r[15])
        : "r"(taddr)
        : "memory");
#pragma unroll
    for (int i = 0; i < 16; ++i) v[i] = __uint_as_float(r[i]);
}

// tcgen05.st of 16 columns (32 lanes x 32 bit) from registers; complete after tmem_st_wait.
__device__ __forceinline__ void tmem_st16(uint32_t taddr, const float (&v)[16]) {
    asm volatile(
        "tcgen05.st.sync.aligned.32x32b.x16.b32 [%0], "
        "{%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,%16};" ::"r"(taddr),
        "f"(v[0]), "f"(v[1]), "f"(v[2]), "f"(v[3]), "f"(v[4]), "f"(v[5]), "f"(v[6]), "f"(v[7]),
        "f"(v[8]), "f"(v[9]), "f"(v[10]), "f"(v[11]), "f"(v[12]), "f"(v[13]), "f"(v[14]), "f"(v[15])
        : "memory");
}

__device__ __forceinline__ void tmem_st_wait() {
    asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory");
}

__device__ __forceinline__ void tmem_ld_wait() {
    asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
}

__device__ __forceinline__ void reg_fence(float (&v)[16]) {
    asm volatile(""
                 : "+f"(v[0]), "+f"(v[1]), "+f"(v[2]), "+f"(v[3]), "+f"(v[4]), "+f"(v[5]),
                   "+f"(v[6]), "+f"(v[7]), "+f"(v[8]), "+f"(v[9]), "+f"(v[10]), "+f"(v[11]),
                   "+f"(v[12]), "+f"(v[13]), "+f"(v[14]), "+f"(v[15]));
}

// Pass-1 update of 16 columns of one key: d = x * sl2 - max; when some d exceeds the lazy
// threshold the column's sum is rescaled to the new maximum (rare: a column's first visible
// key, or a logit 2^60 above the reference); then sum += 2^d.  MASKED keeps only the columns
// whose window row r = (C0 + i) mod W_PAD satisfies r >= jr (the row sees the key).
template <bool MASKED, int W_PAD, int C0>
__device__ __forceinline__ void stats_block(const float (&v)[16], float* nm, float* s, float sl2,
                                            int jr) {
    float d[16];
#pragma unroll
    for (int i = 0; i < 16; i += 2) fma2(d[i], d[i + 1], v[i], v[i + 1], sl2, sl2, nm[i], nm[i + 1]);
    if (MASKED) {
#pragma unroll
        for (int i = 0; i < 16; ++i) d[i] = ((C0 + i) % W_PAD) >= jr ? d[i] : -INFINITY;
    }
    if (max16(d) > kLazyTau) {
#pragma unroll
        for (int i = 0; i < 16; ++i) {
            if (d[i] > kLazyTau) {
                s[i] *= ex2_approx(-d[i]);
                nm[i] = -(v[i] * sl2);
                d[i] = 0.f;
            }
        }
    }
    float e[16];
#pragma unroll
    for (int i = 0; i < 16; ++i) e[i] = ex2_approx(d[i]);
#pragma unroll
    for (int i = 0; i < 16; i += 2) add2(s[i], s[i + 1], s[i], s[i + 1], e[i], e[i + 1]);
}

// Pass-2 sums of one key: per head slot of the MMA's columns, the sum over its rows of
// 2^(x * sl2 - lse).  nlse holds -lse per column (-inf for a column without a real row);
// MASKED keeps only the columns whose window row r = c mod W_PAD satisfies r >= jr.
template <int N, int W_PAD, bool MASKED>
__device__ __forceinline__ void prob_sums(const float (&vv)[N / 16][16], float sl2, const float* nlse,
                                          int jr, float (&accum)[N / W_PAD]) {
    constexpr int kHeads = N / W_PAD;
    constexpr int kPiece = W_PAD < 16 ? W_PAD : 16;  // a head's columns in one 16-column chunk
    float acc2[kHeads][2];
#pragma unroll
    for (int h = 0; h < kHeads; ++h) acc2[h][0] = acc2[h][1] = 0.f;
#pragma unroll
    for (int hh = 0; hh < N / 16; ++hh) {
        float nl[16];
#pragma unroll
        for (int q = 0; q < 4; ++q) {
            const float4 x = reinterpret_cast<const float4*>(nlse + 16 * hh)[q];
            nl[4 * q] = x.x;
            nl[4 * q + 1] = x.y;
            nl[4 * q + 2] = x.z;
            nl[4 * q + 3] = x.w;
        }
        float d[16];
#pragma unroll
        for (int i = 0; i < 16; i += 2)
            fma2(d[i], d[i + 1], vv[hh][i], vv[hh][i + 1], sl2, sl2, nl[i], nl[i + 1]);
        if (MASKED) {
#pragma unroll
            for (int i = 0; i < 16; ++i) d[i] = ((16 * hh + i) % W_PAD) >= jr ? d[i] : -INFINITY;
        }
#pragma unroll
        for (int i = 0; i < 16; ++i) d[i] = ex2_approx(d[i]);
#pragma unroll
        for (int q = 0; q < 16 / kPiece; ++q) {
            float* x = d + q * kPiece;
            pair_tree<kPiece>(x);
            const int h = (16 * hh + q * kPiece) / W_PAD;
            add2(acc2[h][0], acc2[h][1], acc2[h][0], acc2[h][1], x[0], x[1]);
        }
    }
#pragma unroll
    for (int h = 0; h < kHeads; ++h) accum[h] = acc2[h][0] + acc2[h][1];
}


// End of a pass-1 item for one warpgroup of kCols columns: per column, the warp maximum by
// redux and the sums rescaled to it, the warps' sums by recursive halving, then the four
// warps through shared memory `red` (128 pairs); thread c < kCols stores column c's
// (max, sum) at out[c] once the publisher has released the previous use of this
// pub_full/pub_empty pair (phase `pub_phase`), and arrives on pub_full.
__device__ __forceinline__ bool item_partials(float (&m)[kCols], float (&s)[kCols], float2* red, int eq,
                                              int lane, int wtid, uint64_t* gbar, uint32_t& gphase,
                                              uint64_t* pub_full, uint64_t* pub_empty, uint32_t pub_phase,
                                              float2* out, volatile int* abort, long long lim) {
#pragma unroll
    for (int i = 0; i < kCols; ++i) {
        const float M = redux_max(m[i]);
        s[i] *= ex2_approx(m[i] - M);
        m[i] = M;
    }
    transpose_reduce<kCols>(s, m, lane);  // lane l: column l
    red[eq * 32 + lane] = make_float2(m[0], s[0]);
    if (!group_sync(gbar, gphase, abort, lim)) return false;
    if (wtid < kCols) {
        float M = red[wtid].x;
#pragma unroll
        for (int q = 1; q < 4; ++q) M = fmaxf(M, red[q * 32 + wtid].x);
        float S = 0.f;
#pragma unroll
        for (int q = 0; q < 4; ++q) {
            const float2 x = red[q * 32 + wtid];
            S += x.y * ex2_approx(x.x - M);
        }
        if (!mbar_wait(pub_empty, pub_phase ^ 1, abort, lim)) return false;
        out[wtid] = make_float2(M, S);
        mbar_arrive(pub_full);
    }
    return true;
}

template <int N>
__device__ __forceinline__ bool unit_combine(const ScoreParams& p, const ScoreUnit& U, int wtid,
                                             uint64_t* gbar, uint32_t& gphase, float2* red_b,
                                             float* nlse, uint64_t colmask, volatile int* abort,
                                             long long lim);

// The unit's lse per column, for the pass-2 warpgroup (128 threads): thread 0 waits (bounded
// acquire spin) until every item of the unit has published its partials, then the warpgroup
// combines them -- column pairs by 16-byte loads, the items split over kParts groups of
// threads, up to kU loads in flight per thread -- and writes -lse per column to nlse (-inf
// for a column without a real window row or without a visible key).
template <int N>
__device__ __forceinline__ bool unit_lse(const ScoreParams& p, const ScoreUnit& U, int unit, int wtid,
                                         uint64_t* gbar, uint32_t& gphase, volatile int* verdict,
                                         float2* red_b, float* nlse, uint64_t colmask,
                                         volatile int* abort, long long lim) {
    constexpr int kNW = N / kCols;
    if (wtid == 0) {
        const int target = U.nitems * kNW;
        const long long t0 = clock64();
        bool got = true;
        for (uint32_t k = 1; ld_acquire(p.counters + unit) < target; ++k) {
            __nanosleep(64);
            if ((k & 63u) == 0u && (*abort || clock64() - t0 > lim)) {
                got = false;
                break;
            }
        }
        verdict[0] = got ? 1 : 0;  // the acquire load orders the reads of the partials below
    }
    if (!group_sync(gbar, gphase, abort, lim) || verdict[0] == 0) return false;
    return unit_combine<N>(p, U, wtid, gbar, gphase, red_b, nlse, colmask, abort, lim);
}

// The combining part of unit_lse, for a warpgroup that already knows (by an acquire, carried
// to it by a CTA-scope barrier) that every item of the unit has published its partials.
template <int N>
__device__ __forceinline__ bool unit_combine(const ScoreParams& p, const ScoreUnit& U, int wtid,
                                             uint64_t* gbar, uint32_t& gphase, float2* red_b,
                                             float* nlse, uint64_t colmask, volatile int* abort,
                                             long long lim) {
    constexpr int kPairs = N / 2, kParts = 128 / kPairs, kU = 20;
    static_assert(kParts * N <= 256, "red_b holds 256 entries");
    const int c2 = wtid % kPairs, part = wtid / kPairs;
    float M0 = -INFINITY, S0 = 0.f, M1 = -INFINITY, S1 = 0.f;
    const float4* src = reinterpret_cast<const float4*>(p.partials + static_cast<size_t>(U.first_item) * N) + c2;
    for (int k0 = part; k0 < U.nitems; k0 += kParts * kU) {
        float4 pr[kU];
#pragma unroll
        for (int u = 0; u < kU; ++u) {
            const int k = k0 + u * kParts;
            pr[u] = k < U.nitems ? __ldcg(src + static_cast<size_t>(k) * kPairs)
                                 : make_float4(-INFINITY, 0.f, -INFINITY, 0.f);
        }
#pragma unroll
        for (int u = 0; u < kU; ++u) {
            float Mn = fmaxf(M0, pr[u].x);
            if (Mn > -INFINITY) {
                S0 = S0 * ex2_approx(M0 - Mn) + pr[u].y * ex2_approx(pr[u].x - Mn);
                M0 = Mn;
            }
            Mn = fmaxf(M1, pr[u].z);
            if (Mn > -INFINITY) {
                S1 = S1 * ex2_approx(M1 - Mn) + pr[u].w * ex2_approx(pr[u].z - Mn);
                M1 = Mn;
            }
        }
    }
    red_b[part * N + 2 * c2] = make_float2(M0, S0);
    red_b[part * N + 2 * c2 + 1] = make_float2(M1, S1);
    if (!group_sync(gbar, gphase, abort, lim)) return false;
    if (wtid < N) {  // part 0 always holds item 0, so M2 turns finite first
        float M2 = -INFINITY, S2 = 0.f;
#pragma unroll
        for (int q = 0; q < kParts; ++q) {
            const float2 x = red_b[q * N + wtid];
            const float Mn = fmaxf(M2, x.x);
            S2 = S2 * ex2_approx(M2 - Mn) + x.y * ex2_approx(x.x - Mn);
            M2 = Mn;
        }
        nlse[wtid] = ((colmask >> wtid) & 1u) && S2 > 0.f ? -(M2 + lg2_approx(S2)) : -INFINITY;
    }
    return group_sync(gbar, gphase, abort, lim);
}

// Resident variant (score_resident.cu): launch of one (N, W_PAD) instance.
cudaError_t launch_resident(const ScoreParams& p, int n_cols, int w_pad, int grid, cudaStream_t st);
// Single pass with the rows' lse given (score_lse.cu).
cudaError_t launch_given_lse(const ScoreParams& p, int n_cols, int w_pad, int grid, cudaStream_t st);

}  // namespace ckv
