// Window-attention scoring (arxiv 2508.02401, Sec. 3.3 with the attention of Eq. 2):
//
//   a_h[j] = sum_{r < w, j <= P+r} exp(s_{h,r,j} - lse_{h,r}),   s_{h,r,j} = scale * q_{h,r}.k_j
//
// for every selected head h of a KV group, every window row r and every key j of a sequence
// (P = L - w).  A row's normaliser lse needs every key before any probability can be summed
// over rows, so each key tile is used twice -- once for the row statistics, once for the
// probabilities -- and kept in shared memory in between.
//
// One cooperative launch; one CTA per SM, 384 threads, warp-specialised:
//   warp 0      TMA producer: 128-key x 128-dim bf16 tiles of K (two 128-byte-swizzled boxes of
//               64 dims) into a ring of kSlots shared-memory slots; tile i of an item lives
//               in slot (base + i) % kSlots, base advancing by the item's tile count;
//   warp 1      allocates TMEM and issues tcgen05.mma (M = 128 keys, N = the window rows of a
//               batch of heads, K = 128) into kAccBufs TMEM accumulators;
//   warps 2-3   stage the unit's window query rows (the MMA's B operand);
//   warps 4-11  two epilogue warpgroups, each owning half of the window-row columns; every
//               thread owns one key (one TMEM lane), so per-row running statistics (pass 1)
//               and per-key sums over rows (pass 2) are thread-local.
//
// Work: a unit is (sequence, batch of selected heads of one KV group); its key tiles are cut
// into items (chunks).  Per item:
//   pass 1  tiles in increasing order: per-thread running (max, sum of 2^(x - max)) per row,
//           rescaled only when a logit exceeds the running max by more than 2^8; then the
//           CTA's per-row partial goes to global memory and the unit's arrival counter is
//           incremented;
//   wait    until every item of the unit has published its partial (a bounded spin; all CTAs
//           of a launch are co-resident, and a unit's items all belong to one round);
//   pass 2  tiles in decreasing order, so the last kSlots tiles are still resident and only
//           older ones are loaded again: exp2(x - lse) summed over each head's rows.
// Items are dealt out in rounds of gridDim.x; CTA b takes item (round * gridDim.x + b).
#include "ckv_device.cuh"
#include "ckv_internal.h"

#include <string.h>

#include <mutex>

namespace ckv {

constexpr int kSlots = 6;
constexpr int kTileBytes = kTileKeys * kHeadDim * 2;  // 32 KiB
constexpr int kHalfBytes = kTileBytes / 2;            // 64 dims x 128 keys
// The running maximum of a row is only moved when a logit exceeds it by more than 2^60: the
// running sum then stays far below the fp32 range (at most keys * 2^60), and terms that are
// 2^-126 below the reference are negligible against the reference term itself.
constexpr float kLazyTau = 60.0f;
constexpr int kEpiWG = 4;                             // epilogue warpgroups
constexpr int kAccBufs = 4;                           // TMEM accumulators (MMA runs ahead)
constexpr int kEpiThreads = 128 * kEpiWG;
constexpr int kThreads = 128 + kEpiThreads;

struct alignas(128) ScoreParams {
    CUtensorMap tmap_k;            // K as {128 (dim), H_kv, T}, box {64, 1, 128}, 128B swizzle
    const __nv_bfloat16* q_win;    // [S, w, H_q, 128] packed
    const int32_t* cu_seqlens;     // device [S+1] (checked against cu_hash)
    float2* partials;              // [n_items, N]: (max, sum) per window-row column
    int* counters;                 // [n_units] arrivals, zero at launch
    float* scores;                 // [n_sel, T]
    int* status;
    int S, T, Hq, w, n_rounds, n_items, n_units;
    uint32_t cu_hash;
    float sl2;                     // softmax scale * log2(e)
    int16_t batch_group[kMaxBatches];   // KV head of each head batch
    int16_t batch_first[kMaxBatches];   // score row of the batch's first head
    int16_t batch_nheads[kMaxBatches];  // heads in the batch
    int16_t sel_heads[kMaxQHeads];      // query head of each score row
    ScoreItem items[kMaxScoreItems];    // [n_rounds * gridDim.x]
    ScoreUnit units[kMaxScoreUnits];
};

template <int N>
struct SmemLayout {
    static constexpr int kQ = kSlots * kTileBytes;
    static constexpr int kQHalf = N * 128;
    static constexpr int kBars = kQ + 2 * kQHalf;
    // full[kSlots], freed[kSlots], acc_full[kAccBufs], acc_empty[kAccBufs], q_full, q_empty, done
    static constexpr int kNumBars = 2 * kSlots + 2 * kAccBufs + 3;
    static constexpr int kRed = kBars + 8 * kNumBars;   // float2 [512] reduction scratch
    static constexpr int kLse = kRed + 8 * 512;         // float [N]
    static constexpr int kXsum = kLse + 4 * N + 16;     // float [2][kEpiWG][128] (lse: N + flag)
    static constexpr int kFills = kXsum + 4 * 2 * kEpiWG * 128;  // int [2][kSlots]
    static constexpr int kTmemSlot = kFills + 4 * 2 * kSlots;
    static constexpr int kAbort = kTmemSlot + 4;
    static constexpr int kBytes = kAbort + 4;
    static constexpr int kDynamic = kBytes + 1024;      // slack to align the base to 1024 B
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

// Sum / max of an array by a balanced tree (short dependency chains).
template <int C>
__device__ __forceinline__ float tree_sum(float (&x)[C]) {
#pragma unroll
    for (int w = C / 2; w >= 1; w >>= 1)
#pragma unroll
        for (int i = 0; i < w; ++i) x[i] += x[i + w];
    return x[0];
}

__device__ __forceinline__ int ld_acquire(const int* p) {
    int v;
    asm volatile("ld.acquire.gpu.global.b32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
    return v;
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

template <int CPW>
__device__ __forceinline__ void tmem_ld_cols(uint32_t taddr, float (&v)[CPW]) {
    if constexpr (CPW == 32) {
        tmem_ld32(taddr, v);
    } else if constexpr (CPW == 16) {
        uint32_t r[16];
        asm volatile(
            "tcgen05.ld.sync.aligned.32x32b.x16.b32 "
            "{%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15}, [%16];\n\t"
            "tcgen05.wait::ld.sync.aligned;"
            : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]),
              "=r"(r[6]), "=r"(r[7]), "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]),
              "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15])
            : "r"(taddr)
            : "memory");
#pragma unroll
        for (int i = 0; i < 16; ++i) v[i] = __uint_as_float(r[i]);
    } else {
        static_assert(CPW == 8, "CPW");
        uint32_t r[8];
        asm volatile(
            "tcgen05.ld.sync.aligned.32x32b.x8.b32 {%0,%1,%2,%3,%4,%5,%6,%7}, [%8];\n\t"
            "tcgen05.wait::ld.sync.aligned;"
            : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]),
              "=r"(r[6]), "=r"(r[7])
            : "r"(taddr)
            : "memory");
#pragma unroll
        for (int i = 0; i < 8; ++i) v[i] = __uint_as_float(r[i]);
    }
}

// Valid-column mask of one thread for a tile: columns holding a real window row that sees
// key j.  Row r of a head sees key j iff r >= j - P (causal window); keys >= L are padding.
template <int CPW, int W_PAD>
__device__ __forceinline__ uint32_t tile_mask(uint32_t colmask, int col0, int t, int j, int P, int L) {
    const bool edge = (t * kTileKeys + kTileKeys - 1 >= P) || (t * kTileKeys + kTileKeys > L);
    if (!edge) return colmask;
    if (j >= L) return 0u;
    const int jr = j - P;
    uint32_t cm = 0;
#pragma unroll
    for (int i = 0; i < CPW; ++i) cm |= (((col0 + i) % W_PAD) >= jr ? 1u : 0u) << i;
    return colmask & cm;
}

template <int N, int W_PAD>
__global__ void __launch_bounds__(kThreads, 1) score_kernel(const __grid_constant__ ScoreParams p) {
    static_assert(N == 32 || N == 64, "N");
    static_assert(W_PAD == 8 || W_PAD == 16 || W_PAD == 32 || W_PAD == 64, "W_PAD");
    static_assert(W_PAD <= N, "a head's rows fit in one MMA");
    constexpr int CPW = N / kEpiWG;                    // columns per epilogue warpgroup
    constexpr int kWgPerHead = W_PAD > CPW ? W_PAD / CPW : 1;
    constexpr bool kSplitHead = kWgPerHead > 1;        // one head spans several warpgroups
    constexpr int HPW = kSplitHead ? 1 : CPW / W_PAD;  // heads (or a part of one) per warpgroup
    using SL = SmemLayout<N>;
    constexpr uint32_t kIdesc = idesc_bf16_f32(kTileKeys, N);
    constexpr uint32_t kFullMask = CPW == 32 ? 0xffffffffu : ((1u << CPW) - 1u);

    extern __shared__ uint8_t smem_raw[];
    uint8_t* sm = reinterpret_cast<uint8_t*>(
        (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
    uint8_t* slots = sm;
    uint8_t* qbuf = sm + SL::kQ;
    uint64_t* bars = reinterpret_cast<uint64_t*>(sm + SL::kBars);
    uint64_t* full = bars;
    uint64_t* freed = bars + kSlots;
    uint64_t* acc_full = bars + 2 * kSlots;
    uint64_t* acc_empty = acc_full + kAccBufs;
    uint64_t* q_full = acc_empty + kAccBufs;
    uint64_t* q_empty = q_full + 1;
    uint64_t* done = q_empty + 1;
    float2* red = reinterpret_cast<float2*>(sm + SL::kRed);
    float* lse_s = reinterpret_cast<float*>(sm + SL::kLse);
    float* xsum = reinterpret_cast<float*>(sm + SL::kXsum);
    int* fills = reinterpret_cast<int*>(sm + SL::kFills);
    uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(sm + SL::kTmemSlot);
    volatile int* abort = reinterpret_cast<volatile int*>(sm + SL::kAbort);

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;

    if (threadIdx.x == 0) {
        for (int i = 0; i < kSlots; ++i) {
            mbar_init(&full[i], 1);
            mbar_init(&freed[i], 1);
        }
        for (int i = 0; i < kAccBufs; ++i) {
            mbar_init(&acc_full[i], 1);
            mbar_init(&acc_empty[i], kEpiThreads / 32);  // one arrival per epilogue warp
        }
        mbar_init(q_full, 64);
        mbar_init(q_empty, 1);
        mbar_init(done, 1);
        for (int i = 0; i < 2 * kSlots; ++i) fills[i] = 0;
        *abort = 0;
        fence_mbar_init();
        tma_prefetch_desc(&p.tmap_k);
    }
    if (warp == 1) {
        tmem_alloc(tmem_slot, kAccBufs * N);
        tmem_relinquish();
    }
    if (blockIdx.x == 0 && threadIdx.x == 64 && seqlens_hash(p.cu_seqlens, p.S) != p.cu_hash)
        record_error(p.status, kDevBadSeqlens, 100);
    tc_fence_before_sync();
    __syncthreads();
    tc_fence_after_sync();
    const uint32_t tmem_base = *tmem_slot;

    if (warp == 0) {
        // ------------------------------------------------------------ TMA producer
        if (lane == 0) {
            int* pf = fills;  // fills issued per slot
            int base = 0;     // slot of the item's first tile: the ring continues across items
            bool ok = true;
            auto load = [&](const ScoreUnit& U, int tile0, int jt) {
                const int s = (base + jt) % kSlots;
                if (!mbar_wait(&freed[s], (pf[s] & 1) ^ 1, abort)) return false;
                ++pf[s];
                mbar_arrive_expect_tx(&full[s], kTileBytes);
                uint8_t* dst = slots + s * kTileBytes;
                const int tok = U.seq_start + (tile0 + jt) * kTileKeys;
                const int g = p.batch_group[U.batch];
                tma_load_3d(dst, &p.tmap_k, &full[s], 0, g, tok);
                tma_load_3d(dst + kHalfBytes, &p.tmap_k, &full[s], 64, g, tok);
                return true;
            };
            for (int r = 0; ok && r < p.n_rounds; ++r) {
                const ScoreItem& I = p.items[r * gridDim.x + blockIdx.x];
                const int n = I.ntiles;
                if (n == 0) continue;
                const ScoreUnit& U = p.units[I.unit];
                for (int jt = 0; ok && jt < n; ++jt) ok = load(U, I.tile0, jt);               // pass 1
                for (int jt = n - kSlots - 1; ok && jt >= 0; --jt) ok = load(U, I.tile0, jt);  // pass 2
                base = (base + n) % kSlots;
            }
            if (!ok) {
                *abort = 1;
                record_error(p.status, kDevTimeout, 10);
            }
            // Let every issued copy land before the block may exit.
            for (int s = 0; s < kSlots; ++s) {
                volatile int never = 0;
                if (pf[s] > 0) mbar_wait(&full[s], (pf[s] - 1) & 1, &never);
            }
        }
    } else if (warp == 1) {
        // ------------------------------------------------------------ MMA issuer
        if (lane == 0) {
            int* mf = fills + kSlots;  // fills consumed per slot
            int acc_it = 0, item_it = 0, base = 0;
            bool ok = true;
            auto mma_tile = [&](int s, bool wait_fill, bool release) {
                if (wait_fill) {
                    if (!mbar_wait(&full[s], mf[s] & 1, abort)) return false;
                    ++mf[s];
                }
                const int acc = acc_it % kAccBufs;
                if (!mbar_wait(&acc_empty[acc], ((acc_it / kAccBufs) & 1) ^ 1, abort)) return false;
                tc_fence_after_sync();
                const uint32_t d_tmem = tmem_base + static_cast<uint32_t>(acc * N);
                const uint32_t a0 = smem_u32(slots + s * kTileBytes);
                const uint32_t b0 = smem_u32(qbuf);
#pragma unroll
                for (int kk = 0; kk < kHeadDim / 16; ++kk) {
                    const uint32_t koff = (kk & 3) * 32;
                    const uint64_t ad = sdesc_k_major_sw128(a0 + (kk >> 2) * kHalfBytes + koff);
                    const uint64_t bd = sdesc_k_major_sw128(b0 + (kk >> 2) * SL::kQHalf + koff);
                    umma_bf16(d_tmem, ad, bd, kIdesc, kk > 0 ? 1u : 0u);
                }
                umma_commit(&acc_full[acc]);
                if (release) umma_commit(&freed[s]);
                ++acc_it;
                return true;
            };
            for (int r = 0; ok && r < p.n_rounds; ++r) {
                const ScoreItem& I = p.items[r * gridDim.x + blockIdx.x];
                const int n = I.ntiles;
                if (n == 0) continue;
                if (!mbar_wait(q_full, item_it & 1, abort)) {
                    ok = false;
                    break;
                }
                tc_fence_after_sync();
                // pass 1: a tile that is evicted before pass 2 frees its slot right away
                for (int jt = 0; ok && jt < n; ++jt)
                    ok = mma_tile((base + jt) % kSlots, true, jt < n - kSlots);
                // pass 2: resident tiles need no new fill; every tile frees its slot after use
                for (int jt = n - 1; ok && jt >= 0; --jt)
                    ok = mma_tile((base + jt) % kSlots, jt < n - kSlots, true);
                if (!ok) break;
                base = (base + n) % kSlots;
                umma_commit(q_empty);
                ++item_it;
            }
            if (!ok) {
                *abort = 1;
                record_error(p.status, kDevTimeout, 11);
            }
            umma_commit(done);
            volatile int never = 0;
            mbar_wait(done, 0, &never);
        }
        __syncwarp();
    } else if (warp < 4) {
        // ------------------------------------------------------------ query-row staging
        const int tid = threadIdx.x - 64;
        int item_it = 0;
        for (int r = 0; r < p.n_rounds; ++r) {
            const ScoreItem& I = p.items[r * gridDim.x + blockIdx.x];
            if (I.ntiles == 0) continue;
            const ScoreUnit& U = p.units[I.unit];
            if (!mbar_wait(q_empty, (item_it & 1) ^ 1, abort, 500)) {  // a long, idle wait
                *abort = 1;
                record_error(p.status, kDevTimeout, 12);
                break;
            }
            const int first = p.batch_first[U.batch], nheads = p.batch_nheads[U.batch];
            // Each thread owns one 16-byte chunk c of rows r0, r0+4, ...; every load is issued
            // before any store.
            constexpr int kPer = N * 16 / 64;
            const int c = tid & 15, r0 = tid >> 4;
            uint4 vals[kPer];
#pragma unroll
            for (int i = 0; i < kPer; ++i) {
                const int row = r0 + 4 * i;
                const int slot = row / W_PAD, rr = row % W_PAD;
                vals[i] = make_uint4(0u, 0u, 0u, 0u);
                if (slot < nheads && rr < p.w) {
                    const int h = p.sel_heads[first + slot];
                    const uint4* src = reinterpret_cast<const uint4*>(
                        p.q_win + ((static_cast<size_t>(U.seq) * p.w + rr) * p.Hq + h) * kHeadDim);
                    vals[i] = __ldg(src + c);
                }
            }
#pragma unroll
            for (int i = 0; i < kPer; ++i) {
                const int row = r0 + 4 * i;
                const int half = c >> 3, cc = c & 7;
                *reinterpret_cast<uint4*>(qbuf + half * SL::kQHalf + row * 128 +
                                          ((cc ^ (row & 7)) << 4)) = vals[i];
            }
            fence_proxy_async_smem();
            mbar_arrive(q_full);
            ++item_it;
        }
    } else {
        // ------------------------------------------------------------ epilogue
        const int wg = (warp - 4) >> 2;      // warpgroup: columns [wg*CPW, wg*CPW+CPW)
        const int eq = warp & 3;             // TMEM lane quarter
        const int etid = threadIdx.x - 128;  // 0 .. kEpiThreads-1 over the warpgroups
        const int col0 = wg * CPW;
        const uint32_t lane_base = static_cast<uint32_t>(eq * 32) << 16;
        int acc_it = 0;
        bool ok = true;
        for (int r = 0; ok && r < p.n_rounds; ++r) {
            const int item = r * gridDim.x + blockIdx.x;
            // Everything the loops need, copied out of the parameter tables once (asm with a
            // memory clobber inside the loops would otherwise force reloads).
            const ScoreItem I = p.items[item];
            const int n = I.ntiles;
            if (n == 0) continue;
            const ScoreUnit U = p.units[I.unit];
            const int L = U.len, P = L - p.w;
            const int first = p.batch_first[U.batch], nheads = p.batch_nheads[U.batch];
            const int T = p.T;
            const float sl2 = p.sl2;
            float* const scores = p.scores;
            uint32_t colmask = 0;  // this warpgroup's columns that hold a real window row
#pragma unroll
            for (int i = 0; i < CPW; ++i) {
                const int c = col0 + i;
                if ((c % W_PAD) < p.w && (c / W_PAD) < nheads) colmask |= 1u << i;
            }
            float st_a[CPW];  // pass 1: running max (log2 units); pass 2: lse (log2 units)
            float st_b[CPW];  // pass 1: running sum relative to st_a

            // ---------------------------------------------------- pass 1
            for (int jt = 0; jt < n; ++jt, ++acc_it) {
                const int acc = acc_it % kAccBufs;
                if (!mbar_wait(&acc_full[acc], (acc_it / kAccBufs) & 1, abort)) {
                    ok = false;
                    break;
                }
                tc_fence_after_sync();
                float v[CPW];
                tmem_ld_cols<CPW>(tmem_base + lane_base + static_cast<uint32_t>(acc * N + col0), v);
                tc_fence_before_sync();
                __syncwarp();
                if (lane == 0) mbar_arrive(&acc_empty[acc]);
                const int t = I.tile0 + jt;
                const int j = t * kTileKeys + eq * 32 + lane;  // sequence-local key
                const uint32_t vm = tile_mask<CPW, W_PAD>(colmask, col0, t, j, P, L);
                if (jt == 0) {
                    // The thread's first key of the item seeds each row's running maximum.  A
                    // row that cannot see this key cannot see the thread's later keys either.
#pragma unroll
                    for (int i = 0; i < CPW; ++i) {
                        const bool valid = (vm >> i) & 1u;
                        st_a[i] = valid ? v[i] * sl2 : -1e30f;
                        st_b[i] = valid ? 1.f : 0.f;
                    }
                    continue;
                }
                if (vm == kFullMask) {
#pragma unroll
                    for (int i = 0; i < CPW; ++i) v[i] = fmaf(v[i], sl2, -st_a[i]);
                } else {
#pragma unroll
                    for (int i = 0; i < CPW; ++i) {
                        const float d = fmaf(v[i], sl2, -st_a[i]);
                        v[i] = ((vm >> i) & 1u) ? d : -INFINITY;
                    }
                }
                float dm[CPW / 4];  // max by a short tree
#pragma unroll
                for (int i = 0; i < CPW / 4; ++i)
                    dm[i] = fmaxf(fmaxf(v[4 * i], v[4 * i + 1]), fmaxf(v[4 * i + 2], v[4 * i + 3]));
#pragma unroll
                for (int w = CPW / 8; w >= 1; w >>= 1)
#pragma unroll
                    for (int i = 0; i < w; ++i) dm[i] = fmaxf(dm[i], dm[i + w]);
                const float dmax = dm[0];
                if (dmax > kLazyTau) {  // a new running maximum well above the old one
#pragma unroll
                    for (int i = 0; i < CPW; ++i) {
                        if (v[i] > kLazyTau) {
                            st_b[i] *= ex2_approx(-v[i]);
                            st_a[i] += v[i];
                            v[i] = 0.f;
                        }
                    }
                }
#pragma unroll
                for (int i = 0; i < CPW; ++i) st_b[i] += ex2_approx(v[i]);
            }
            if (!ok) break;

            // The warpgroup's 128 threads per column: warp max by redux, rescale to it, warp sums
            // by recursive halving; then the 4 warps of each warpgroup through shared memory.
#pragma unroll
            for (int i = 0; i < CPW; ++i) {
                const float M = redux_max(st_a[i]);
                st_b[i] *= ex2_approx(st_a[i] - M);
                st_a[i] = M;
            }
            transpose_reduce<CPW>(st_b, st_a, lane);
            {
                constexpr int kLanesPerCol = 32 / CPW;
                if (lane % kLanesPerCol == 0)
                    red[(wg * 4 + eq) * CPW + lane / kLanesPerCol] = make_float2(st_a[0], st_b[0]);
            }
            named_bar_sync(1, kEpiThreads);
            if (etid < N) {
                const int cw = etid / CPW, ci = etid % CPW;
                float M = red[(cw * 4) * CPW + ci].x;
#pragma unroll
                for (int q = 1; q < 4; ++q) M = fmaxf(M, red[(cw * 4 + q) * CPW + ci].x);
                float S = 0.f;
#pragma unroll
                for (int q = 0; q < 4; ++q) {
                    const float2 x = red[(cw * 4 + q) * CPW + ci];
                    S += x.y * ex2_approx(x.x - M);
                }
                p.partials[static_cast<size_t>(item) * N + etid] = make_float2(M, S);
            }
            named_bar_sync(1, kEpiThreads);

            // ---------------------------------------------------- exchange with the unit
            if (etid == 0) {
                // The barrier above orders the block's partial stores before this thread's
                // release; the fence makes that release cumulative at GPU scope.
                __threadfence();
                red_release_add(p.counters + I.unit, 1);
                const long long t0 = clock64();
                bool got = true;
                for (uint32_t it = 1; ld_acquire(p.counters + I.unit) < U.nitems; ++it) {
                    __nanosleep(64);
                    if ((it & 63u) == 0u && (*abort || clock64() - t0 > kWaitTimeoutCycles)) {
                        *abort = 1;
                        record_error(p.status, kDevTimeout, 13);
                        got = false;
                        break;
                    }
                }
                __threadfence();
                lse_s[N] = got ? 1.f : 0.f;  // one verdict for the whole epilogue
            }
            named_bar_sync(1, kEpiThreads);
            if (lse_s[N] == 0.f) {
                ok = false;
                break;
            }
            {
                // All epilogue threads: column etid % N, items part, part + parts, ...
                constexpr int kParts = kEpiThreads / N;
                const int c = etid % N, part = etid / N;
                float M = -INFINITY, S = 0.f;
                const float2* src = p.partials + static_cast<size_t>(U.first_item) * N + c;
                for (int k = part; k < U.nitems; k += kParts) {
                    const float2 pr = __ldcg(src + static_cast<size_t>(k) * N);
                    const float Mn = fmaxf(M, pr.x);
                    S = S * ex2_approx(M - Mn) + pr.y * ex2_approx(pr.x - Mn);
                    M = Mn;
                }
                red[part * N + c] = make_float2(M, S);
                named_bar_sync(1, kEpiThreads);
                if (etid < N) {
                    float M2 = -INFINITY, S2 = 0.f;
#pragma unroll
                    for (int q = 0; q < kParts; ++q) {
                        const float2 x = red[q * N + etid];
                        const float Mn = fmaxf(M2, x.x);
                        S2 = S2 * ex2_approx(M2 - Mn) + x.y * ex2_approx(x.x - Mn);
                        M2 = Mn;
                    }
                    lse_s[etid] = M2 + lg2_approx(S2);
                }
            }
            named_bar_sync(1, kEpiThreads);
#pragma unroll
            for (int i = 0; i < CPW; ++i) st_a[i] = lse_s[col0 + i];

            // ---------------------------------------------------- pass 2 (tiles in reverse)
            for (int jt = n - 1; jt >= 0; --jt, ++acc_it) {
                const int acc = acc_it % kAccBufs;
                if (!mbar_wait(&acc_full[acc], (acc_it / kAccBufs) & 1, abort)) {
                    ok = false;
                    break;
                }
                tc_fence_after_sync();
                float v[CPW];
                tmem_ld_cols<CPW>(tmem_base + lane_base + static_cast<uint32_t>(acc * N + col0), v);
                tc_fence_before_sync();
                __syncwarp();
                if (lane == 0) mbar_arrive(&acc_empty[acc]);
                const int t = I.tile0 + jt;
                const int j = t * kTileKeys + eq * 32 + lane;
                const uint32_t vm = tile_mask<CPW, W_PAD>(colmask, col0, t, j, P, L);
                if (vm == kFullMask) {
#pragma unroll
                    for (int i = 0; i < CPW; ++i) v[i] = ex2_approx(fmaf(v[i], sl2, -st_a[i]));
                } else {
#pragma unroll
                    for (int i = 0; i < CPW; ++i) {
                        const float e = ex2_approx(fmaf(v[i], sl2, -st_a[i]));
                        v[i] = ((vm >> i) & 1u) ? e : 0.f;
                    }
                }
                // per-head sums by trees over each head's (up to W_PAD) columns
                constexpr int kSeg = kSplitHead ? CPW : W_PAD;
                float accum[HPW];
#pragma unroll
                for (int h = 0; h < HPW; ++h) {
                    float seg[kSeg];
#pragma unroll
                    for (int i = 0; i < kSeg; ++i) seg[i] = v[h * kSeg + i];
                    accum[h] = tree_sum<kSeg>(seg);
                }
                const bool key_ok = j < L;
                const size_t col = static_cast<size_t>(U.seq_start) + j;
                if constexpr (kSplitHead) {
                    // the head's first warpgroup adds the other warpgroups' parts
                    float* xs = xsum + (acc & 1) * kEpiWG * 128;
                    const int part = wg % kWgPerHead, hg = wg / kWgPerHead;
                    if (part != 0) xs[wg * 128 + eq * 32 + lane] = accum[0];
                    named_bar_sync(2, kEpiThreads);
                    if (part == 0 && key_ok && hg < nheads) {
                        float sum = accum[0];
#pragma unroll
                        for (int q = 1; q < kWgPerHead; ++q) sum += xs[(wg + q) * 128 + eq * 32 + lane];
                        scores[static_cast<size_t>(first + hg) * T + col] = sum;
                    }
                } else if (key_ok) {
#pragma unroll
                    for (int h = 0; h < HPW; ++h) {
                        const int hg = wg * HPW + h;
                        if (hg < nheads) scores[static_cast<size_t>(first + hg) * T + col] = accum[h];
                    }
                }
            }
        }
        if (!ok) {
            *abort = 1;
            record_error(p.status, kDevTimeout, 14);
        }
    }

    tc_fence_before_sync();
    __syncthreads();
    if (warp == 1) {
        tc_fence_after_sync();
        tmem_dealloc(tmem_base, kAccBufs * N);
    }
}

// ------------------------------------------------------------------------------ host side
namespace {

template <int N, int W_PAD>
cudaError_t launch_one(const ScoreParams& p, int grid, cudaStream_t stream) {
    auto kern = score_kernel<N, W_PAD>;
    constexpr int smem = SmemLayout<N>::kDynamic;
    static bool configured = false;  // benign race: the attribute call is idempotent
    if (!configured) {
        cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
        if (e != cudaSuccess) return e;
        configured = true;
    }
    cudaLaunchConfig_t cfg;
    memset(&cfg, 0, sizeof cfg);
    cfg.gridDim = dim3(grid);
    cfg.blockDim = dim3(kThreads);
    cfg.dynamicSmemBytes = smem;
    cfg.stream = stream;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeCooperative;  // all CTAs co-resident: the unit waits need it
    attr[0].val.cooperative = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, kern, p);
}

cudaError_t dispatch(const ScoreParams& p, int n_cols, int w_pad, int grid, cudaStream_t st) {
    if (n_cols == 32) {
        if (w_pad == 8) return launch_one<32, 8>(p, grid, st);
        if (w_pad == 16) return launch_one<32, 16>(p, grid, st);
        if (w_pad == 32) return launch_one<32, 32>(p, grid, st);
    } else if (n_cols == 64) {
        if (w_pad == 8) return launch_one<64, 8>(p, grid, st);
        if (w_pad == 16) return launch_one<64, 16>(p, grid, st);
        if (w_pad == 32) return launch_one<64, 32>(p, grid, st);
        if (w_pad == 64) return launch_one<64, 64>(p, grid, st);
    }
    return cudaErrorInvalidValue;
}

}  // namespace

cudaError_t launch_score(const ScoreLaunch& L, cudaStream_t stream) {
    static_assert(sizeof(ScoreParams) <= 32000, "kernel parameters");
    static ScoreParams p;  // ~25 KB, kept off the host stack; calls are serialised by `mu`
    static std::mutex mu;
    std::lock_guard<std::mutex> lock(mu);
    memset(&p, 0, sizeof(p));
    p.tmap_k = L.tmap_k;
    p.q_win = reinterpret_cast<const __nv_bfloat16*>(L.q_win);
    p.cu_seqlens = L.cu_seqlens_dev;
    p.partials = reinterpret_cast<float2*>(L.partials);
    p.counters = L.counters;
    p.scores = L.scores;
    p.status = L.status;
    p.S = L.S;
    p.T = L.T;
    p.Hq = L.Hq;
    p.w = L.w;
    p.cu_hash = L.cu_hash;
    p.sl2 = L.softmax_scale * 1.4426950408889634f;
    for (int b = 0; b < L.nb; ++b) {
        p.batch_group[b] = static_cast<int16_t>(L.batch_group[b]);
        p.batch_first[b] = static_cast<int16_t>(L.batch_first[b]);
        p.batch_nheads[b] = static_cast<int16_t>(L.batch_nheads[b]);
    }
    for (int i = 0; i < L.n_sel; ++i) p.sel_heads[i] = static_cast<int16_t>(L.sel_heads[i]);
    // One launch per slice of rounds whose items and units fit the parameter tables.
    for (const ScoreSlice& sl : L.slices) {
        p.n_rounds = sl.n_rounds;
        p.n_items = sl.n_rounds * L.grid;
        p.n_units = sl.n_units;
        memcpy(p.items, L.items.data() + sl.item0, sizeof(ScoreItem) * p.n_items);
        memcpy(p.units, L.units.data() + sl.unit0, sizeof(ScoreUnit) * p.n_units);
        cudaError_t e = cudaMemsetAsync(L.counters, 0, sizeof(int) * sl.n_units, stream);
        if (e != cudaSuccess) return e;
        e = dispatch(p, L.n_cols, L.w_pad, L.grid, stream);
        if (e != cudaSuccess) return e;
    }
    return cudaSuccess;
}

}  // namespace ckv
