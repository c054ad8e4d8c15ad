// Window-attention scoring with the window rows' log-sum-exp given by the caller (arxiv
// 2508.02401, Sec. 3.3 with the attention of Eq. 2):
//
//   a_h[j] = sum_{r < w, j <= P+r} exp(s_{h,r,j} - lse_{h,r}),   s_{h,r,j} = scale * q_{h,r}.k_j,
//
// where lse_{h,r} = log sum_{j <= P+r} exp(s_{h,r,j}) is the normaliser that a prefill
// attention kernel computes anyway for every query row.  With it given, the scores need one
// pass over K and no exchange between CTAs: each key tile is read, multiplied and turned into
// its probabilities once, so the work splits evenly over the CTAs (a CTA's run of tiles may
// cross sequences and head batches).
//
// One CTA per SM, 512 threads:
//   warp 0       producer: per work item, TMA loads of the window query rows into one of two
//                buffers, then of its key tiles into a ring of kRing slots (evict-first);
//   warp 1       allocates all 512 TMEM columns and issues tcgen05.mma (M = 128 keys, N window
//                rows, K = 128) of tile u of the CTA into accumulator u mod (512 / N), once the
//                epilogue has released it;
//   warps 4-15   three epilogue warpgroups; tile u goes to warpgroup u mod 3, which reads its
//                N columns from TMEM, releases the accumulator, and sums 2^(x - lse) over each
//                head's rows.
#include "score_layers.cuh"

#include <string.h>

namespace ckv {
namespace {

constexpr int kQB = 2;       // query-row buffers
constexpr int kEpiWG = 3;    // epilogue warpgroups

template <int N>
struct LseLayout {
    static constexpr int kSlots = 512 / N;              // TMEM accumulators
    static constexpr int kRing = 6;                     // key-tile ring
    static constexpr int kQBytes = N * 256;
    static constexpr int kQHalf = N * 128;
    static constexpr int kRingOff = 0;
    static constexpr int kQ = kRingOff + kRing * kTileBytes;
    static constexpr int kBars = kQ + kQB * kQBytes;
    static constexpr int kFull = 0, kFree = kFull + kRing, kTFull = kFree + kRing,
                         kTEmpty = kTFull + kSlots, kQFull = kTEmpty + kSlots, kQEmpty = kQFull + kQB,
                         kDone = kQEmpty + kQB, kGroup = kDone + 1, kNumBars = kGroup + kEpiWG;
    static constexpr int kTmemSlot = kBars + 8 * kNumBars;
    static constexpr int kAbort = kTmemSlot + 4;
    static constexpr int kBytes = kAbort + 4;
    static constexpr int kDynamic = kBytes + 1024;      // slack to align the base to 1024 B
};
// dynamic + the kernel's static shared memory (under 1 KB) within the 227 KB a block may use
static_assert(LseLayout<64>::kDynamic + 1024 <= 232448, "shared memory, N = 64");
static_assert(LseLayout<32>::kDynamic + 1024 <= 232448, "shared memory, N = 32");

template <int N, int W_PAD>
__global__ void __launch_bounds__(kThreads, 1) score_lse_kernel(const __grid_constant__ ScoreParams p) {
    static_assert(N == 32 || N == 64, "N");
    static_assert(W_PAD == 8 || W_PAD == 16 || W_PAD == 32 || W_PAD == 64, "W_PAD");
    static_assert(W_PAD <= N, "a head's rows fit in one MMA");
    using SL = LseLayout<N>;
    constexpr int kSlots = SL::kSlots, kRing = SL::kRing;
    constexpr uint32_t kIdesc = idesc_bf16_f32(kTileKeys, N);
    constexpr int kHeads = N / W_PAD;

    extern __shared__ uint8_t smem_raw[];
    uint8_t* sm = reinterpret_cast<uint8_t*>(
        (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
    uint8_t* ring = sm + SL::kRingOff;
    uint8_t* qbuf = sm + SL::kQ;
    uint64_t* bars = reinterpret_cast<uint64_t*>(sm + SL::kBars);
    uint64_t* full = bars + SL::kFull;
    uint64_t* freed = bars + SL::kFree;
    uint64_t* t_full = bars + SL::kTFull;
    uint64_t* t_empty = bars + SL::kTEmpty;
    uint64_t* q_full = bars + SL::kQFull;
    uint64_t* q_empty = bars + SL::kQEmpty;
    uint64_t* done = bars + SL::kDone;
    uint64_t* group = bars + SL::kGroup;
    __shared__ __align__(16) float nlse_s[kEpiWG][64];  // per epilogue warpgroup: -lse (log2)
    uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(sm + SL::kTmemSlot);
    volatile int* abort = reinterpret_cast<volatile int*>(sm + SL::kAbort);

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;

    if (threadIdx.x == 0) {
        for (int i = 0; i < kRing; ++i) {
            mbar_init(&full[i], 1);
            mbar_init(&freed[i], 1);
        }
        for (int i = 0; i < kSlots; ++i) {
            mbar_init(&t_full[i], 1);
            mbar_init(&t_empty[i], 4);  // the four warps of the tile's warpgroup
        }
        for (int i = 0; i < kQB; ++i) {
            mbar_init(&q_full[i], 1);
            mbar_init(&q_empty[i], 1);
        }
        mbar_init(done, 1);
        for (int i = 0; i < kEpiWG; ++i) mbar_init(&group[i], kGroupArrivals);
        *abort = 0;
        fence_mbar_init();
        tma_prefetch_desc(&p.tmap_k);
        tma_prefetch_desc(&p.tmap_q);
    }
    // Query slots of head batches with fewer heads than the MMA's columns are never loaded;
    // zeros there keep those (unused) columns finite.
    for (int i = threadIdx.x; i < kQB * SL::kQBytes / 16; i += kThreads)
        reinterpret_cast<uint4*>(qbuf)[i] = make_uint4(0u, 0u, 0u, 0u);
    fence_proxy_async_smem();
    if (warp == 1) {
        tmem_alloc(tmem_slot, 512);
        tmem_relinquish();
    }
    if (blockIdx.x == 0 && threadIdx.x == 64 && seqlens_hash(p.cu_seqlens, p.S) != p.cu_hash)
        record_error(p.status, kDevBadSeqlens, 100);
    tc_fence_before_sync();
    __syncthreads();
    tc_fence_after_sync();
    const uint32_t tmem_base = *tmem_slot;
    // Registers: launched at 128 per thread; the control warpgroup gives up to 56, which lets
    // the three epilogue warpgroups take 152 each (128*56 + 384*152 = 65536).
    const int R = p.n_rounds;
    const int G = gridDim.x;
    const long long lim = p.wait_cycles;
    auto item_of = [&](int r) -> const ScoreItem& { return p.items[r * G + blockIdx.x]; };

    if (warp < kWarpA) {
        setmaxnreg_dec<56>();
        if (warp == 0) {
            // ------------------------------------------------------------ TMA producer
            if (lane == 0) {
                const uint64_t policy = l2_policy_evict_first();
                int use = 0, it = 0;
                bool ok = true;
                for (int r = 0; ok && r < R; ++r) {
                    const ScoreItem& I = item_of(r);
                    const int n = I.ntiles;
                    if (n == 0) continue;
                    const ScoreUnit& U = p.units[I.unit];
                    const int g = p.batch_group[U.batch];
                    const int qb = it % kQB;
                    if (!mbar_wait(&q_empty[qb], ((it / kQB) & 1) ^ 1, abort, lim)) {
                        ok = false;
                        break;
                    }
                    uint8_t* qdst = qbuf + qb * SL::kQBytes;
                    const int first_row = p.batch_first[U.batch], nheads = p.batch_nheads[U.batch];
                    mbar_arrive_expect_tx(&q_full[qb], static_cast<uint32_t>(nheads * W_PAD * 256));
                    for (int slot = 0; slot < nheads; ++slot) {
                        const int h = p.sel_heads[first_row + slot];
                        uint8_t* d = qdst + slot * W_PAD * 128;
                        tma_load_3d(d, &p.tmap_q, &q_full[qb], 0, h, U.seq * p.w);
                        tma_load_3d(d + SL::kQHalf, &p.tmap_q, &q_full[qb], 64, h, U.seq * p.w);
                    }
                    for (int jt = 0; ok && jt < n; ++jt, ++use) {
                        const int s = use % kRing;
                        if (!mbar_wait(&freed[s], ((use / kRing) & 1) ^ 1, abort, lim)) {
                            ok = false;
                            break;
                        }
                        mbar_arrive_expect_tx(&full[s], kTileBytes);
                        uint8_t* dst = ring + s * kTileBytes;
                        const int tok = U.seq_start + (I.tile0 + jt) * kTileKeys;
                        tma_load_3d_hint(dst, &p.tmap_k, &full[s], 0, g, tok, policy);
                        tma_load_3d_hint(dst + kHalfBytes, &p.tmap_k, &full[s], 64, g, tok, policy);
                    }
                    ++it;
                }
                if (!ok) {
                    *abort = 1;
                    record_error(p.status, kDevTimeout, 30);
                }
                for (int k = (use > kRing ? use - kRing : 0); k < use; ++k) {
                    volatile int never = 0;
                    mbar_wait(&full[k % kRing], (k / kRing) & 1, &never);
                }
                for (int k = (it > kQB ? it - kQB : 0); k < it; ++k) {
                    volatile int never = 0;
                    mbar_wait(&q_full[k % kQB], (k / kQB) & 1, &never);
                }
            }
        } else if (warp == 1) {
            // ------------------------------------------------------------ MMA issuer
            if (lane == 0) {
                int use = 0, it = 0;
                bool ok = true;
                for (int r = 0; ok && r < R; ++r) {
                    const ScoreItem& I = item_of(r);
                    const int n = I.ntiles;
                    if (n == 0) continue;
                    const int qb = it % kQB;
                    if (!mbar_wait(&q_full[qb], (it / kQB) & 1, abort, lim)) {
                        ok = false;
                        break;
                    }
                    tc_fence_after_sync();
                    const uint32_t b0 = smem_u32(qbuf + qb * SL::kQBytes);
                    for (int jt = 0; jt < n; ++jt, ++use) {
                        const int s = use % kRing, acc = use % kSlots;
                        if (!mbar_wait(&t_empty[acc], ((use / kSlots) & 1) ^ 1, abort, lim) ||
                            !mbar_wait(&full[s], (use / kRing) & 1, abort, lim)) {
                            ok = false;
                            break;
                        }
                        tc_fence_after_sync();
                        const uint32_t a0 = smem_u32(ring + s * kTileBytes);
                        const uint32_t d_tmem = tmem_base + static_cast<uint32_t>(acc * N);
#pragma unroll
                        for (int kk = 0; kk < kHeadDim / 16; ++kk) {
                            const uint32_t koff = (kk & 3) * 32;
                            const uint64_t ad = sdesc_k_major_sw128(a0 + (kk >> 2) * kHalfBytes + koff);
                            const uint64_t bd = sdesc_k_major_sw128(b0 + (kk >> 2) * SL::kQHalf + koff);
                            umma_bf16(d_tmem, ad, bd, kIdesc, kk > 0 ? 1u : 0u);
                        }
                        umma_commit(&t_full[acc]);
                        umma_commit(&freed[s]);
                    }
                    if (!ok) break;
                    umma_commit(&q_empty[qb]);
                    ++it;
                }
                if (!ok) {
                    *abort = 1;
                    record_error(p.status, kDevTimeout, 31);
                }
                umma_commit(done);
                volatile int never = 0;
                mbar_wait(done, 0, &never);
            }
            __syncwarp();
        }
    } else {
        // ------------------------------------------------------------ epilogue
        setmaxnreg_inc<152>();
        const int e = (warp - kWarpA) >> 2;  // this warpgroup takes the CTA's tiles u = e mod 3
        const int eq = warp & 3;
        const int wtid = threadIdx.x - (kWarpA + 4 * e) * 32;
        const uint32_t lane_base = static_cast<uint32_t>(eq * 32) << 16;
        uint64_t* gbar = &group[e];
        uint32_t gphase = 0;
        float* nl = nlse_s[e];
        const float sl2 = p.sl2;
        int use = 0;
        bool ok = true;
        for (int r = 0; ok && r < R; ++r) {
            const ScoreItem I = p.items[r * G + blockIdx.x];
            const int n = I.ntiles;
            if (n == 0) continue;
            const int j0 = ((e - use) % kEpiWG + kEpiWG) % kEpiWG;  // this warpgroup's first tile
            if (j0 < n) {
                const ScoreUnit U = p.units[I.unit];
                const int L = U.len, P = L - p.w;
                const int first = p.batch_first[U.batch], nheads = p.batch_nheads[U.batch];
                // -lse per column in log2 units: -inf for a column without a real window row,
                // or whose row's query position is before the sequence start (L < w)
                if (!group_sync(gbar, gphase, abort, lim)) {  // the previous item's values are read
                    ok = false;
                    break;
                }
                if (wtid < N) {
                    const int h = wtid / W_PAD, row = wtid % W_PAD;
                    float v = -INFINITY;
                    if (h < nheads && row < p.w && P + row >= 0) {
                        const int qh = p.sel_heads[first + h];
                        const float x = __ldg(p.lse + static_cast<size_t>(qh) * p.lse_stride +
                                              static_cast<size_t>(U.seq) * p.w + row);
                        v = -x * 1.4426950408889634f;
                    }
                    nl[wtid] = v;
                }
                if (!group_sync(gbar, gphase, abort, lim)) {
                    ok = false;
                    break;
                }
                for (int jt = j0; jt < n; jt += kEpiWG) {
                    const int u = use + jt, acc = u % kSlots;
                    if (!__all_sync(0xffffffffu, mbar_wait(&t_full[acc], (u / kSlots) & 1, abort, lim))) {
                        ok = false;
                        break;
                    }
                    tc_fence_after_sync();
                    const int t = I.tile0 + jt;
                    const int j = t * kTileKeys + eq * 32 + lane;
                    const bool edge = (t * kTileKeys + kTileKeys - 1 >= P) || (t * kTileKeys + kTileKeys > L);
                    const uint32_t taddr = tmem_base + lane_base + static_cast<uint32_t>(acc * N);
                    float vv[N / 16][16];
#pragma unroll
                    for (int hh = 0; hh < N / 16; ++hh) tmem_ld16_nowait(taddr + hh * 16, vv[hh]);
                    tmem_ld_wait();
#pragma unroll
                    for (int hh = 0; hh < N / 16; ++hh) reg_fence(vv[hh]);
                    tc_fence_before_sync();
                    __syncwarp();
                    if (lane == 0) mbar_arrive(&t_empty[acc]);  // the accumulator is free
                    float accum[kHeads];
                    if (!edge) {
                        prob_sums<N, W_PAD, false>(vv, sl2, nl, 0, accum);
                    } else {  // row r sees key j iff r >= j - P; keys past L are padding
                        prob_sums<N, W_PAD, true>(vv, sl2, nl, j < L ? j - P : (1 << 30), accum);
                    }
                    if (j < L) {
                        const size_t col = static_cast<size_t>(U.seq_start) + j;
#pragma unroll
                        for (int h = 0; h < kHeads; ++h)
                            if (h < nheads) p.scores[static_cast<size_t>(first + h) * p.T + col] = accum[h];
                    }
                }
            }
            use += n;
        }
        if (!ok) {
            *abort = 1;
            record_error(p.status, kDevTimeout, 32);
        }
    }

    tc_fence_before_sync();
    __syncthreads();
    if (warp == 1) {
        tc_fence_after_sync();
        tmem_dealloc(tmem_base, 512);
    }
}

template <int N, int W_PAD>
cudaError_t launch_lse(const ScoreParams& p, int grid, cudaStream_t stream) {
    auto kern = score_lse_kernel<N, W_PAD>;
    constexpr int smem = LseLayout<N>::kDynamic;
    static bool configured = false;  // benign race: the attribute call is idempotent
    if (!configured) {
        cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
        if (e != cudaSuccess) return e;
        configured = true;
    }
    NvtxRange range("score_lse_kernel");
    kern<<<grid, kThreads, smem, stream>>>(p);
    return cudaGetLastError();
}


// ---------------------------------------------------------------- many layers in one launch
// The same single pass over every (layer, head batch, sequence) unit of a multi-layer launch:
// the units' key tiles are cut into items of balanced length (the work items of the two-pass
// multi-layer kernel), and each CTA takes its next item from a global counter when its query
// buffer is free, so that the faster SMs take more of the work and a launch over many layers
// ends with at most one item of imbalance.  With no exchange between CTAs no wait crosses a
// CTA, and the launch needs no co-residency.  Roles as above; the producer posts each item
// index into a ring that the MMA warp and every epilogue warp read.
constexpr int kLseItemRing = 8;

template <int N>
struct LseLayersLayout {
    using B = LseLayout<N>;
    static constexpr int kSlots = B::kSlots, kRing = B::kRing, kQBytes = B::kQBytes, kQHalf = B::kQHalf;
    static constexpr int kRingOff = 0;
    static constexpr int kQ = kRingOff + kRing * kTileBytes;
    static constexpr int kBars = kQ + kQB * kQBytes;
    static constexpr int kFull = 0, kFree = kFull + kRing, kTFull = kFree + kRing,
                         kTEmpty = kTFull + kSlots, kQFull = kTEmpty + kSlots, kQEmpty = kQFull + kQB,
                         kDone = kQEmpty + kQB, kGroup = kDone + 1, kItemFull = kGroup + kEpiWG,
                         kItemFree = kItemFull + kLseItemRing, kNumBars = kItemFree + kLseItemRing;
    static constexpr int kItems = kBars + 8 * kNumBars;  // int[kLseItemRing]: posted item indices
    static constexpr int kTmemSlot = kItems + 4 * kLseItemRing;
    static constexpr int kAbort = kTmemSlot + 4;
    static constexpr int kBytes = kAbort + 4;
    static constexpr int kDynamic = kBytes + 1024;
};
static_assert(LseLayersLayout<64>::kDynamic + 1024 <= 232448, "shared memory, N = 64");
static_assert(LseLayersLayout<32>::kDynamic + 1024 <= 232448, "shared memory, N = 32");
// Readers of a posted item index: the MMA issuer and the twelve epilogue warps.
constexpr int kItemReaders = 1 + 4 * kEpiWG;

template <int N, int W_PAD>
__global__ void __launch_bounds__(kThreads, 1) score_lse_layers_kernel(const __grid_constant__ LayersParams p) {
    static_assert(N == 32 || N == 64, "N");
    static_assert(W_PAD == 8 || W_PAD == 16 || W_PAD == 32 || W_PAD == 64, "W_PAD");
    static_assert(W_PAD <= N, "a head's rows fit in one MMA");
    using SL = LseLayersLayout<N>;
    constexpr int kSlots = SL::kSlots, kRing = SL::kRing;
    constexpr uint32_t kIdesc = idesc_bf16_f32(kTileKeys, N);
    constexpr int kHeads = N / W_PAD;

    extern __shared__ uint8_t smem_raw[];
    uint8_t* sm = reinterpret_cast<uint8_t*>(
        (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
    uint8_t* ring = sm + SL::kRingOff;
    uint8_t* qbuf = sm + SL::kQ;
    uint64_t* bars = reinterpret_cast<uint64_t*>(sm + SL::kBars);
    uint64_t* full = bars + SL::kFull;
    uint64_t* freed = bars + SL::kFree;
    uint64_t* t_full = bars + SL::kTFull;
    uint64_t* t_empty = bars + SL::kTEmpty;
    uint64_t* q_full = bars + SL::kQFull;
    uint64_t* q_empty = bars + SL::kQEmpty;
    uint64_t* done = bars + SL::kDone;
    uint64_t* group = bars + SL::kGroup;
    uint64_t* item_full = bars + SL::kItemFull;  // items[k] holds the CTA's next item index
    uint64_t* item_free = bars + SL::kItemFree;  // every reader has read items[k]
    int* items = reinterpret_cast<int*>(sm + SL::kItems);
    __shared__ __align__(16) float nlse_s[kEpiWG][64];  // per epilogue warpgroup: -lse (log2)
    uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(sm + SL::kTmemSlot);
    volatile int* abort = reinterpret_cast<volatile int*>(sm + SL::kAbort);

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int n_items = p.n_items;

    if (threadIdx.x == 0) {
        for (int i = 0; i < kRing; ++i) {
            mbar_init(&full[i], 1);
            mbar_init(&freed[i], 1);
        }
        for (int i = 0; i < kSlots; ++i) {
            mbar_init(&t_full[i], 1);
            mbar_init(&t_empty[i], 4);  // the four warps of the tile's warpgroup
        }
        for (int i = 0; i < kQB; ++i) {
            mbar_init(&q_full[i], 1);
            mbar_init(&q_empty[i], 1);
        }
        mbar_init(done, 1);
        for (int i = 0; i < kEpiWG; ++i) mbar_init(&group[i], kGroupArrivals);
        for (int i = 0; i < kLseItemRing; ++i) {
            mbar_init(&item_full[i], 1);
            mbar_init(&item_free[i], kItemReaders);
        }
        *abort = 0;
        fence_mbar_init();
    }
    if (warp == 0 && lane < p.n_layers) {  // every layer's tensor maps, one lane each
        tma_prefetch_desc(&p.tmap_k[lane]);
        tma_prefetch_desc(&p.tmap_q[lane]);
    }
    // Query slots of head batches with fewer heads than the MMA's columns are never loaded;
    // zeros there keep those (unused) columns finite.
    for (int i = threadIdx.x; i < kQB * SL::kQBytes / 16; i += kThreads)
        reinterpret_cast<uint4*>(qbuf)[i] = make_uint4(0u, 0u, 0u, 0u);
    fence_proxy_async_smem();
    if (warp == 1) {
        tmem_alloc(tmem_slot, 512);
        tmem_relinquish();
    }
    if (blockIdx.x == 0 && threadIdx.x == 64 && seqlens_hash(p.cu_seqlens, p.S_all) != p.cu_hash)
        record_error(p.status, kDevBadSeqlens, 100);
    tc_fence_before_sync();
    __syncthreads();
    tc_fence_after_sync();
    const uint32_t tmem_base = *tmem_slot;
    // Registers as in the one-layer kernel: 128*56 + 384*152 = 65536.
    const long long lim = p.wait_cycles;

    if (warp < kWarpA) {
        setmaxnreg_dec<56>();
        if (warp == 0) {
            // ------------------------------------------------------------ TMA producer
            if (lane == 0) {
                const uint64_t policy = l2_policy_evict_first();
                int* next_item = p.counters + p.n_units;
                int use = 0, it = 0;
                bool ok = true;
                for (;; ++it) {
                    // the next item once its query buffer and its ring entry are free
                    const int qb = it % kQB, k = it % kLseItemRing;
                    if (!mbar_wait(&q_empty[qb], ((it / kQB) & 1) ^ 1, abort, lim) ||
                        !mbar_wait(&item_free[k], ((it / kLseItemRing) & 1) ^ 1, abort, lim)) {
                        ok = false;
                        break;
                    }
                    const int gi = atomicAdd(next_item, 1);
                    items[k] = gi < n_items ? gi : -1;
                    mbar_arrive(&item_full[k]);  // releases items[k] to the other roles
                    if (gi >= n_items) break;
                    const Item I = get_item(p, gi);
                    const int g = p.batch_group[I.batch];
                    const int nheads = p.batch_nheads[I.batch], sel0 = p.batch_sel[I.batch];
                    const CUtensorMap* qm = &p.tmap_q[I.layer];
                    const CUtensorMap* km = &p.tmap_k[I.layer];
                    uint8_t* qdst = qbuf + qb * SL::kQBytes;
                    mbar_arrive_expect_tx(&q_full[qb], static_cast<uint32_t>(nheads * W_PAD * 256));
                    const int row = (p.seq0 + I.seq) * p.w;
                    for (int slot = 0; slot < nheads; ++slot) {
                        const int h = p.sel_heads[sel0 + slot];
                        uint8_t* d = qdst + slot * W_PAD * 128;
                        tma_load_3d(d, qm, &q_full[qb], 0, h, row);
                        tma_load_3d(d + SL::kQHalf, qm, &q_full[qb], 64, h, row);
                    }
                    for (int jt = 0; jt < I.ntiles; ++jt, ++use) {
                        const int s = use % kRing;
                        if (!mbar_wait(&freed[s], ((use / kRing) & 1) ^ 1, abort, lim)) {
                            ok = false;
                            break;
                        }
                        mbar_arrive_expect_tx(&full[s], kTileBytes);
                        uint8_t* dst = ring + s * kTileBytes;
                        const int tok = I.start + (I.tile0 + jt) * kTileKeys;
                        tma_load_3d_hint(dst, km, &full[s], 0, g, tok, policy);
                        tma_load_3d_hint(dst + kHalfBytes, km, &full[s], 64, g, tok, policy);
                    }
                    if (!ok) {
                        ++it;  // its query rows were issued
                        break;
                    }
                }
                if (!ok) {
                    *abort = 1;
                    record_error(p.status, kDevTimeout, 33);
                }
                // let every issued copy land before the block may exit
                volatile int never = 0;
                for (int k = (use > kRing ? use - kRing : 0); k < use; ++k)
                    mbar_wait(&full[k % kRing], (k / kRing) & 1, &never);
                for (int k = (it > kQB ? it - kQB : 0); k < it; ++k)
                    mbar_wait(&q_full[k % kQB], (k / kQB) & 1, &never);
            }
        } else if (warp == 1) {
            // ------------------------------------------------------------ MMA issuer
            if (lane == 0) {
                int use = 0;
                bool ok = true;
                for (int it = 0;; ++it) {
                    int gi = -1;
                    if (!wait_item<kLseItemRing>(item_full, items, it, &gi, abort, lim)) {
                        ok = false;
                        break;
                    }
                    mbar_arrive(&item_free[it % kLseItemRing]);
                    if (gi < 0) break;
                    const int n = get_item(p, gi).ntiles;
                    const int qb = it % kQB;
                    if (!mbar_wait(&q_full[qb], (it / kQB) & 1, abort, lim)) {
                        ok = false;
                        break;
                    }
                    tc_fence_after_sync();
                    const uint32_t b0 = smem_u32(qbuf + qb * SL::kQBytes);
                    for (int jt = 0; jt < n; ++jt, ++use) {
                        const int s = use % kRing, acc = use % kSlots;
                        if (!mbar_wait(&t_empty[acc], ((use / kSlots) & 1) ^ 1, abort, lim) ||
                            !mbar_wait(&full[s], (use / kRing) & 1, abort, lim)) {
                            ok = false;
                            break;
                        }
                        tc_fence_after_sync();
                        const uint32_t a0 = smem_u32(ring + s * kTileBytes);
                        const uint32_t d_tmem = tmem_base + static_cast<uint32_t>(acc * N);
#pragma unroll
                        for (int kk = 0; kk < kHeadDim / 16; ++kk) {
                            const uint32_t koff = (kk & 3) * 32;
                            const uint64_t ad = sdesc_k_major_sw128(a0 + (kk >> 2) * kHalfBytes + koff);
                            const uint64_t bd = sdesc_k_major_sw128(b0 + (kk >> 2) * SL::kQHalf + koff);
                            umma_bf16(d_tmem, ad, bd, kIdesc, kk > 0 ? 1u : 0u);
                        }
                        umma_commit(&t_full[acc]);
                        umma_commit(&freed[s]);
                    }
                    if (!ok) break;
                    umma_commit(&q_empty[qb]);
                }
                if (!ok) {
                    *abort = 1;
                    record_error(p.status, kDevTimeout, 34);
                }
                umma_commit(done);
                volatile int never = 0;
                mbar_wait(done, 0, &never);
            }
            __syncwarp();
        }
    } else {
        // ------------------------------------------------------------ epilogue
        setmaxnreg_inc<152>();
        const int e = (warp - kWarpA) >> 2;  // this warpgroup takes the CTA's tiles u = e mod 3
        const int eq = warp & 3;
        const int wtid = threadIdx.x - (kWarpA + 4 * e) * 32;
        const uint32_t lane_base = static_cast<uint32_t>(eq * 32) << 16;
        uint64_t* gbar = &group[e];
        uint32_t gphase = 0;
        float* nl = nlse_s[e];
        const float sl2 = p.sl2;
        const size_t T = static_cast<size_t>(p.T);
        int use = 0;
        bool ok = true;
        for (int it = 0; ok; ++it) {
            int gi = -1, good = 1;
            if (lane == 0) {
                good = wait_item<kLseItemRing>(item_full, items, it, &gi, abort, lim) ? 1 : 0;
                mbar_arrive(&item_free[it % kLseItemRing]);
            }
            gi = __shfl_sync(0xffffffffu, gi, 0);
            if (__shfl_sync(0xffffffffu, good, 0) == 0) {
                ok = false;
                break;
            }
            if (gi < 0) break;
            const Item I = get_item(p, gi);
            const int n = I.ntiles;
            const int j0 = ((e - use) % kEpiWG + kEpiWG) % kEpiWG;  // this warpgroup's first tile
            if (j0 < n) {
                const int L = I.len, P = L - p.w;
                const int nheads = p.batch_nheads[I.batch], sel0 = p.batch_sel[I.batch];
                // the batch's first score row, at the sequence's first token
                float* const out = p.scores[I.layer] + static_cast<size_t>(p.batch_first[I.batch]) * T + I.start;
                // -lse per column in log2 units: -inf for a column without a real window row,
                // or whose row's query position is before the sequence start (L < w)
                if (!group_sync(gbar, gphase, abort, lim)) {  // the previous item's values are read
                    ok = false;
                    break;
                }
                if (wtid < N) {
                    const int h = wtid / W_PAD, row = wtid % W_PAD;
                    float v = -INFINITY;
                    if (h < nheads && row < p.w && P + row >= 0) {
                        const int qh = p.sel_heads[sel0 + h];
                        const float x = __ldg(p.lse[I.layer] + static_cast<size_t>(qh) * p.lse_stride[I.layer] +
                                              static_cast<size_t>(p.seq0 + I.seq) * p.w + row);
                        v = -x * 1.4426950408889634f;
                    }
                    nl[wtid] = v;
                }
                if (!group_sync(gbar, gphase, abort, lim)) {
                    ok = false;
                    break;
                }
                for (int jt = j0; jt < n; jt += kEpiWG) {
                    const int u = use + jt, acc = u % kSlots;
                    if (!__all_sync(0xffffffffu, mbar_wait(&t_full[acc], (u / kSlots) & 1, abort, lim))) {
                        ok = false;
                        break;
                    }
                    tc_fence_after_sync();
                    const int t = I.tile0 + jt;
                    const int j = t * kTileKeys + eq * 32 + lane;
                    const bool edge = (t * kTileKeys + kTileKeys - 1 >= P) || (t * kTileKeys + kTileKeys > L);
                    const uint32_t taddr = tmem_base + lane_base + static_cast<uint32_t>(acc * N);
                    float vv[N / 16][16];
#pragma unroll
                    for (int hh = 0; hh < N / 16; ++hh) tmem_ld16_nowait(taddr + hh * 16, vv[hh]);
                    tmem_ld_wait();
#pragma unroll
                    for (int hh = 0; hh < N / 16; ++hh) reg_fence(vv[hh]);
                    tc_fence_before_sync();
                    __syncwarp();
                    if (lane == 0) mbar_arrive(&t_empty[acc]);  // the accumulator is free
                    float accum[kHeads];
                    if (!edge) {
                        prob_sums<N, W_PAD, false>(vv, sl2, nl, 0, accum);
                    } else {  // row r sees key j iff r >= j - P; keys past L are padding
                        prob_sums<N, W_PAD, true>(vv, sl2, nl, j < L ? j - P : (1 << 30), accum);
                    }
                    if (j < L) {
#pragma unroll
                        for (int h = 0; h < kHeads; ++h)
                            if (h < nheads) out[h * T + j] = accum[h];
                    }
                }
            }
            use += n;
        }
        if (!ok) {
            *abort = 1;
            record_error(p.status, kDevTimeout, 35);
        }
    }

    tc_fence_before_sync();
    __syncthreads();
    if (warp == 1) {
        tc_fence_after_sync();
        tmem_dealloc(tmem_base, 512);
    }
}

template <int N, int W_PAD>
cudaError_t launch_lse_layers(const LayersParams& p, int grid, cudaStream_t stream) {
    auto kern = score_lse_layers_kernel<N, W_PAD>;
    constexpr int smem = LseLayersLayout<N>::kDynamic;
    static bool configured = false;  // benign race: the attribute call is idempotent
    if (!configured) {
        cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
        if (e != cudaSuccess) return e;
        configured = true;
    }
    NvtxRange range("score_lse_layers_kernel");
    kern<<<grid, kThreads, smem, stream>>>(p);
    return cudaGetLastError();
}

}  // namespace

cudaError_t launch_given_lse(const ScoreParams& p, int n_cols, int w_pad, int grid, cudaStream_t st) {
    if (n_cols == 32) {
        if (w_pad == 8) return launch_lse<32, 8>(p, grid, st);
        if (w_pad == 16) return launch_lse<32, 16>(p, grid, st);
        if (w_pad == 32) return launch_lse<32, 32>(p, grid, st);
    } else if (n_cols == 64) {
        if (w_pad == 8) return launch_lse<64, 8>(p, grid, st);
        if (w_pad == 16) return launch_lse<64, 16>(p, grid, st);
        if (w_pad == 32) return launch_lse<64, 32>(p, grid, st);
        if (w_pad == 64) return launch_lse<64, 64>(p, grid, st);
    }
    return cudaErrorInvalidValue;
}

cudaError_t dispatch_lse_layers(const LayersParams& p, int n_cols, int w_pad, int grid, cudaStream_t st) {
    if (n_cols == 32) {
        if (w_pad == 8) return launch_lse_layers<32, 8>(p, grid, st);
        if (w_pad == 16) return launch_lse_layers<32, 16>(p, grid, st);
        if (w_pad == 32) return launch_lse_layers<32, 32>(p, grid, st);
    } else if (n_cols == 64) {
        if (w_pad == 8) return launch_lse_layers<64, 8>(p, grid, st);
        if (w_pad == 16) return launch_lse_layers<64, 16>(p, grid, st);
        if (w_pad == 32) return launch_lse_layers<64, 32>(p, grid, st);
        if (w_pad == 64) return launch_lse_layers<64, 64>(p, grid, st);
    }
    return cudaErrorInvalidValue;
}

}  // namespace ckv
