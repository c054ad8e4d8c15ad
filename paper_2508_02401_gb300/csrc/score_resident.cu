// Window-attention scoring with the logits resident in tensor memory (arxiv 2508.02401,
// Sec. 3.3 with the attention of Eq. 2): the same scores as score_kernel.cu,
//
//   a_h[j] = sum_{r < w, j <= P+r} exp(s_{h,r,j} - lse_{h,r}),   s_{h,r,j} = scale * q_{h,r}.k_j,
//
// for work items short enough that all of an item's key tiles fit in TMEM (512 columns: 512 / N
// tiles of 128 keys x N window-row columns).  Each key tile is read from HBM and multiplied once.
// Pass 1 turns the tile's fp32 logits into exponentials 2^(x - m) in place, m being a reference
// per column that is the same for the 32 keys of a warp (moved, warp-uniformly, only when a
// logit exceeds it by 2^60), and accumulates the row statistics.  After the unit's exchange,
// pass 2 needs no exponential per element: one factor 2^(m - lse) per (warp, column) turns the
// stored values into probabilities.  Without a second read of K, the shared memory goes to a
// deeper ring of key tiles, which keeps more of HBM's latency covered.
//
// One cooperative launch, one CTA per SM, 512 threads:
//   warp 0       producer: per item, TMA loads of the window query rows into one of two
//                buffers, then of its key tiles into a ring of kRing slots (evict-first: each
//                tile is read once);
//   warp 1       allocates all 512 TMEM columns and issues tcgen05.mma (M = 128 keys, N window
//                rows, K = 128) of tile u of the CTA into accumulator u mod (512 / N), once
//                pass 2 has released that accumulator;
//   warp 3       publisher: once an item's pass-1 partials are stored, one release on the
//                unit's arrival counter;
//   warps 4-11   pass 1, one warpgroup per 32 columns; at the end of an item the warps'
//                references go to shared memory;
//   warps 12-15  pass 2: once every item of the unit has published (a bounded acquire spin),
//                the unit's lse, the factors, then per tile the head sums of the products.
// An item's accumulators stay allocated from its MMA until its pass 2, so the next item's
// MMAs use the accumulators it leaves free while this CTA waits for the rest of the unit, and
// the ring keeps loading meanwhile.
#include "score_common.cuh"

#include <mutex>

#include <string.h>

namespace ckv {
namespace {

constexpr int kQB = 2;  // query-row buffers

template <int N>
struct ResLayout {
    static constexpr int kSlots = 512 / N;              // TMEM accumulators
    static constexpr int kRing = N == 64 ? 5 : 6;       // key-tile ring (shared memory)
    static constexpr int kQBytes = N * 256;             // one item's rows: N x 128 bf16
    static constexpr int kQHalf = N * 128;              // 64 dims of them
    static constexpr int kRingOff = 0;
    static constexpr int kQ = kRingOff + kRing * kTileBytes;
    static constexpr int kBars = kQ + kQB * kQBytes;
    static constexpr int kFull = 0, kFree = kFull + kRing, kTFull = kFree + kRing,
                         kTEmpty = kTFull + kSlots, kQFull = kTEmpty + kSlots, kQEmpty = kQFull + kQB,
                         kDone = kQEmpty + kQB, kGroup = kDone + 1,  // A0 A1 B
                         kPubFull = kGroup + 3, kPubEmpty = kPubFull + 2, kMEmpty = kPubEmpty + 2,
                         kNumBars = kMEmpty + 2;
    static constexpr int kTmemSlot = kBars + 8 * kNumBars;
    static constexpr int kAbort = kTmemSlot + 4;
    static constexpr int kBytes = kAbort + 4;
    static constexpr int kDynamic = kBytes + 1024;      // slack to align the base to 1024 B
};
// dynamic + the kernel's static shared memory (under 10 KB) within the 227 KB a block may use
static_assert(ResLayout<64>::kDynamic + 10240 <= 232448, "shared memory, N = 64");
static_assert(ResLayout<32>::kDynamic + 10240 <= 232448, "shared memory, N = 32");

// The exponentials a warp stored for 16 columns of the item's tiles t < jt (accumulators
// (use0 + t) mod kSlots, columns from `tcol`), times fac per column: the rare rescale of a
// column's reference within an item.  Out of line, so that its registers do not weigh on the
// common path.
template <int N>
__device__ __noinline__ void rescale_earlier(uint32_t tcol, int use0, int jt, const float* fac) {
    constexpr int kSlots = 512 / N;
    for (int t = 0; t < jt; ++t) {
        const uint32_t a = tcol + static_cast<uint32_t>(((use0 + t) % kSlots) * N);
        float e[16];
        tmem_ld16_nowait(a, e);
        tmem_ld_wait();
        reg_fence(e);
#pragma unroll
        for (int i = 0; i < 16; ++i) e[i] *= fac[i];
        tmem_st16(a, e);
    }
}

// Pass 1 on 16 columns of one key, in place: d = x * sl2 - m with m the warp's reference for
// the column (nm = -m, the same in every lane), 2^d stored back to the tile's accumulator
// columns at `taddr` (the item's tile jt; its first tile is accumulator use0) and added to
// the thread's running sums.  When some lane's d exceeds 2^60 in a column (always so at the
// column's first visible key in the warp), the warp moves that column's reference to the
// warp's largest logit there, rescales the sums and the exponentials stored for the item's
// earlier tiles -- a rare, warp-uniform path.  MASKED keeps only the columns whose window
// row r = (C0 + i) mod W_PAD satisfies r >= jr (the row sees the key).
template <bool MASKED, int N, int W_PAD, int C0>
__device__ __forceinline__ void stats_store(const float (&v)[16], float* nm, float* s, float sl2, int jr,
                                            uint32_t taddr, uint32_t tcol, int use0, int jt) {
    float d[16];
#pragma unroll
    for (int i = 0; i < 16; i += 2) fma2(d[i], d[i + 1], v[i], v[i + 1], sl2, sl2, nm[i], nm[i + 1]);
    if (MASKED) {
#pragma unroll
        for (int i = 0; i < 16; ++i) d[i] = ((C0 + i) % W_PAD) >= jr ? d[i] : -INFINITY;
    }
    if (__any_sync(0xffffffffu, max16(d) > kLazyTau)) {
        float fac[16];
        bool older = false;
#pragma unroll
        for (int i = 0; i < 16; ++i) {
            fac[i] = 1.f;
            if (__any_sync(0xffffffffu, d[i] > kLazyTau)) {
                const bool seen = !MASKED || d[i] > -INFINITY;
                const float M = redux_max(seen ? v[i] * sl2 : -INFINITY);  // the new reference
                fac[i] = ex2_approx(-nm[i] - M);  // 2^(old reference - new reference)
                s[i] *= fac[i];
                older |= nm[i] < 1e29f;           // the column had a reference before this tile
                nm[i] = -M;
                d[i] = seen ? fmaf(v[i], sl2, -M) : -INFINITY;
            }
        }
        if (older) rescale_earlier<N>(tcol + C0, use0, jt, fac);
    }
#pragma unroll
    for (int i = 0; i < 16; ++i) d[i] = ex2_approx(d[i]);
    tmem_st16(taddr, d);
#pragma unroll
    for (int i = 0; i < 16; i += 2) add2(s[i], s[i + 1], s[i], s[i + 1], d[i], d[i + 1]);
}

// The warp's references of 16 columns at the item's first tile: the largest logit of the
// column among the warp's keys that see it (-nm), or the "none yet" value where none does.
template <bool MASKED, int W_PAD, int C0>
__device__ __forceinline__ void init_refs(const float (&v)[16], float* nm, float sl2, int jr) {
#pragma unroll
    for (int i = 0; i < 16; ++i) {
        const bool seen = !MASKED || ((C0 + i) % W_PAD) >= jr;
        const float M = redux_max(seen ? v[i] * sl2 : -INFINITY);
        nm[i] = M > -INFINITY ? -M : 1e30f;
    }
}

template <int N, int W_PAD>
__global__ void __launch_bounds__(kThreads, 1) score_resident_kernel(const __grid_constant__ ScoreParams p) {
    static_assert(N == 32 || N == 64, "N");
    static_assert(W_PAD == 8 || W_PAD == 16 || W_PAD == 32 || W_PAD == 64, "W_PAD");
    static_assert(W_PAD <= N, "a head's rows fit in one MMA");
    constexpr int kNW = N / kCols;  // pass-1 warpgroups
    using SL = ResLayout<N>;
    constexpr int kSlots = SL::kSlots, kRing = SL::kRing;
    constexpr uint32_t kIdesc = idesc_bf16_f32(kTileKeys, N);

    extern __shared__ uint8_t smem_raw[];
    uint8_t* sm = reinterpret_cast<uint8_t*>(
        (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
    uint8_t* ring = sm + SL::kRingOff;
    uint8_t* qbuf = sm + SL::kQ;
    uint64_t* bars = reinterpret_cast<uint64_t*>(sm + SL::kBars);
    uint64_t* full = bars + SL::kFull;        // ring slot loaded
    uint64_t* freed = bars + SL::kFree;       // ring slot read by its MMA
    uint64_t* t_full = bars + SL::kTFull;     // accumulator written by its MMA
    uint64_t* t_empty = bars + SL::kTEmpty;   // accumulator read by pass 2
    uint64_t* q_full = bars + SL::kQFull;
    uint64_t* q_empty = bars + SL::kQEmpty;
    uint64_t* done = bars + SL::kDone;
    uint64_t* group = bars + SL::kGroup;
    uint64_t* pub_full = bars + SL::kPubFull;
    uint64_t* pub_empty = bars + SL::kPubEmpty;
    uint64_t* m_empty = bars + SL::kMEmpty;   // an item's references read by pass 2
    __shared__ float2 red_a[2][2][128];       // [item parity][warpgroup][warp * 32 + lane]
    __shared__ float2 red_b[256];             // [part * N + column]
    __shared__ __align__(16) float nlse_s[64];
    __shared__ __align__(16) float ref_s[2][4][64];  // [item parity][warp quarter][column]: m
    __shared__ __align__(16) float fac_s[4][64];     // [warp quarter][column]: 2^(m - lse)
    __shared__ volatile int verdict[1];
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
            mbar_init(&t_empty[i], 4);  // one arrival per pass-2 warp
        }
        for (int i = 0; i < kQB; ++i) {
            mbar_init(&q_full[i], 1);
            mbar_init(&q_empty[i], 1);
        }
        mbar_init(done, 1);
        for (int i = 0; i < 3; ++i) mbar_init(&group[i], kGroupArrivals);
        for (int i = 0; i < 2; ++i) {
            mbar_init(&pub_full[i], 32 * kNW);
            mbar_init(&pub_empty[i], 1);
            mbar_init(&m_empty[i], 1);
        }
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
    // Registers as in score_kernel.cu: launched at 128 per thread; the control warpgroup gives
    // up to 56, the pass-1 warpgroups take 160, pass 2 keeps 128.
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
                    // The window query rows: per head of the batch two boxes of 64 dims x
                    // W_PAD rows in the MMA's 128-byte-swizzled layout.  Rows past w (the next
                    // sequence's, or zeros past the end) land in columns that are never read.
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
                    record_error(p.status, kDevTimeout, 20);
                }
                // Let every issued copy land before the block may exit.
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
                    umma_commit(&q_empty[qb]);  // the item's query rows are free
                    ++it;
                }
                if (!ok) {
                    *abort = 1;
                    record_error(p.status, kDevTimeout, 21);
                }
                umma_commit(done);
                volatile int never = 0;
                mbar_wait(done, 0, &never);
            }
            __syncwarp();
        } else if (warp == 3) {
            // ------------------------------------------------------------ publisher
            if (lane == 0) {
                int it = 0;
                for (int r = 0; r < R; ++r) {
                    const ScoreItem& I = item_of(r);
                    if (I.ntiles == 0) continue;
                    if (!mbar_wait(&pub_full[it & 1], (it >> 1) & 1, abort, lim)) {
                        *abort = 1;
                        record_error(p.status, kDevTimeout, 22);
                        break;
                    }
                    red_release_add(p.counters + I.unit, kNW);
                    mbar_arrive(&pub_empty[it & 1]);
                    ++it;
                }
            }
        }
    } else if (warp < kWarpB) {
        // ------------------------------------------------------------ pass 1
        setmaxnreg_inc<160>();
        const int wg = (warp - kWarpA) >> 2;  // columns [wg*32, wg*32+32)
        if (wg < kNW) {
            const int eq = warp & 3;
            const int wtid = threadIdx.x - (kWarpA + 4 * wg) * 32;
            const int col0 = wg * kCols;
            const uint32_t tcol = tmem_base + (static_cast<uint32_t>(eq * 32) << 16) + static_cast<uint32_t>(col0);
            const float sl2 = p.sl2;
            uint64_t* gbar = &group[wg];
            uint32_t gphase = 0;
            int use = 0, a_item = 0;
            bool ok = true;
            for (int r = 0; ok && r < R; ++r) {
                const int item = r * G + blockIdx.x;
                const ScoreItem I = p.items[item];
                const int n = I.ntiles;
                if (n == 0) continue;
                const ScoreUnit U = p.units[I.unit];
                const int L = U.len, P = L - p.w;
                float nm[kCols], sm_[kCols];  // negated warp reference (log2 units), running sum
#pragma unroll
                for (int i = 0; i < kCols; ++i) {
                    nm[i] = 1e30f;
                    sm_[i] = 0.f;
                }
                const int use0 = use;
                bool ready = false;  // this tile's MMA is known to be complete
                for (int jt = 0; jt < n; ++jt, ++use) {
                    const int acc = use % kSlots;
                    // (the warp decides as one: the tcgen05 accesses below are warp-collective)
                    if (!ready && !__all_sync(0xffffffffu, mbar_wait(&t_full[acc], (use / kSlots) & 1, abort, lim))) {
                        ok = false;
                        break;
                    }
                    tc_fence_after_sync();
                    const int t = I.tile0 + jt;
                    const int j = t * kTileKeys + eq * 32 + lane;
                    const bool edge = (t * kTileKeys + kTileKeys - 1 >= P) || (t * kTileKeys + kTileKeys > L);
                    const uint32_t taddr = tcol + static_cast<uint32_t>(acc * N);
                    float vv[2][16];
                    tmem_ld16_nowait(taddr, vv[0]);
                    tmem_ld16_nowait(taddr + 16, vv[1]);
                    // while the loads are in flight: is the next tile's MMA already complete?
                    ready = jt + 1 < n &&
                            __all_sync(0xffffffffu, mbar_test(&t_full[(use + 1) % kSlots], ((use + 1) / kSlots) & 1));
                    tmem_ld_wait();
                    reg_fence(vv[0]);
                    reg_fence(vv[1]);
                    if (!edge) {
                        if (jt == 0) {
                            init_refs<false, W_PAD, 0>(vv[0], nm, sl2, 0);
                            init_refs<false, W_PAD, 16>(vv[1], nm + 16, sl2, 0);
                        }
                        stats_store<false, N, W_PAD, 0>(vv[0], nm, sm_, sl2, 0, taddr, tcol, use0, jt);
                        stats_store<false, N, W_PAD, 16>(vv[1], nm + 16, sm_ + 16, sl2, 0, taddr + 16, tcol, use0, jt);
                    } else {  // row r sees key j iff r >= j - P; keys past L are padding
                        const int jr = (j < L ? j - P : (1 << 30)) - (W_PAD == 64 ? col0 : 0);
                        if (jt == 0) {
                            init_refs<true, W_PAD, 0>(vv[0], nm, sl2, jr);
                            init_refs<true, W_PAD, 16>(vv[1], nm + 16, sl2, jr);
                        }
                        stats_store<true, N, W_PAD, 0>(vv[0], nm, sm_, sl2, jr, taddr, tcol, use0, jt);
                        stats_store<true, N, W_PAD, 16>(vv[1], nm + 16, sm_ + 16, sl2, jr, taddr + 16, tcol, use0, jt);
                    }
                }
                if (!ok) break;
                tmem_st_wait();          // the exponentials are in TMEM before pass 2 may read them
                tc_fence_before_sync();  // and this item's TMEM accesses precede the syncs below
                float m[kCols];
#pragma unroll
                for (int i = 0; i < kCols; ++i) m[i] = -nm[i];
                // the warp's references for pass 2, once it has read those of the item two back
                if (!mbar_wait(&m_empty[a_item & 1], ((a_item >> 1) & 1) ^ 1, abort, lim)) {
                    ok = false;
                    break;
                }
                if (lane == 0) {
                    float4* dst = reinterpret_cast<float4*>(&ref_s[a_item & 1][eq][col0]);
#pragma unroll
                    for (int i = 0; i < kCols; i += 4) dst[i / 4] = make_float4(m[i], m[i + 1], m[i + 2], m[i + 3]);
                }
                if (!item_partials(m, sm_, red_a[a_item & 1][wg], eq, lane, wtid, gbar, gphase,
                                   &pub_full[a_item & 1], &pub_empty[a_item & 1], (a_item >> 1) & 1,
                                   p.partials + static_cast<size_t>(item) * N + col0, abort, lim)) {
                    ok = false;
                    break;
                }
                ++a_item;
            }
            if (!ok) {
                *abort = 1;
                record_error(p.status, kDevTimeout, 23);
            }
            tmem_st_wait();  // no store of this warp is in flight when the block frees TMEM
        }
    } else {
        // ------------------------------------------------------------ pass 2
        const int eq = warp & 3;
        const int wtid = threadIdx.x - kWarpB * 32;
        const uint32_t lane_base = static_cast<uint32_t>(eq * 32) << 16;
        uint64_t* gbar = &group[2];
        uint32_t gphase = 0;
        constexpr int kHeads = N / W_PAD;
        constexpr int kPiece = W_PAD < 16 ? W_PAD : 16;  // a head's columns in one 16-column chunk
        int use = 0, k = 0;
        bool ok = true;
        for (int r = 0; ok && r < R; ++r) {
            const ScoreItem I = p.items[r * G + blockIdx.x];
            const int n = I.ntiles;
            if (n == 0) continue;
            const ScoreUnit U = p.units[I.unit];
            const int L = U.len;
            const int first = p.batch_first[U.batch], nheads = p.batch_nheads[U.batch];
            uint64_t colmask = 0;  // columns that hold a real window row
#pragma unroll
            for (int c = 0; c < N; ++c)
                if ((c % W_PAD) < p.w && (c / W_PAD) < nheads) colmask |= 1ull << c;
            if (!unit_lse<N>(p, U, I.unit, wtid, gbar, gphase, verdict, red_b, nlse_s, colmask, abort, lim)) {
                ok = false;
                break;
            }
            // factors 2^(m - lse) per (pass-1 warp quarter, column); 0 for a column without a
            // real row (-lse = -inf there)
            for (int x = wtid; x < 4 * N; x += 128)
                fac_s[x / N][x % N] = ex2_approx(ref_s[k & 1][x / N][x % N] + nlse_s[x % N]);
            if (!group_sync(gbar, gphase, abort, lim)) {
                ok = false;
                break;
            }
            if (wtid == 0) mbar_arrive(&m_empty[k & 1]);
            // Pass 1 stored the item's exponentials (and waited for the stores) before it
            // published, which the exchange above observed: the TMEM reads below follow them.
            tc_fence_after_sync();
            const float* fq = fac_s[eq];
            for (int jt = 0; jt < n; ++jt, ++use) {
                const int acc = use % kSlots;
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
                float hs[kHeads][2];
#pragma unroll
                for (int h = 0; h < kHeads; ++h) hs[h][0] = hs[h][1] = 0.f;
#pragma unroll
                for (int hh = 0; hh < N / 16; ++hh) {
                    float* e = vv[hh];
#pragma unroll
                    for (int q = 0; q < 4; ++q) {
                        const float4 f = reinterpret_cast<const float4*>(fq + 16 * hh)[q];
                        mul2(e[4 * q], e[4 * q + 1], e[4 * q], e[4 * q + 1], f.x, f.y);
                        mul2(e[4 * q + 2], e[4 * q + 3], e[4 * q + 2], e[4 * q + 3], f.z, f.w);
                    }
#pragma unroll
                    for (int q = 0; q < 16 / kPiece; ++q) {
                        float* y = e + q * kPiece;
                        pair_tree<kPiece>(y);
                        const int h = (16 * hh + q * kPiece) / W_PAD;
                        add2(hs[h][0], hs[h][1], hs[h][0], hs[h][1], y[0], y[1]);
                    }
                }
                const int j = (I.tile0 + jt) * kTileKeys + eq * 32 + lane;
                if (j < L) {
                    const size_t col = static_cast<size_t>(U.seq_start) + j;
#pragma unroll
                    for (int h = 0; h < kHeads; ++h)
                        if (h < nheads) p.scores[static_cast<size_t>(first + h) * p.T + col] = hs[h][0] + hs[h][1];
                }
            }
            ++k;
        }
        if (!ok) {
            *abort = 1;
            record_error(p.status, kDevTimeout, 24);
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
cudaError_t launch_res(const ScoreParams& p, int grid, cudaStream_t stream) {
    auto kern = score_resident_kernel<N, W_PAD>;
    constexpr int smem = ResLayout<N>::kDynamic;
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
    NvtxRange range("score_resident_kernel");
    return cudaLaunchKernelEx(&cfg, kern, p);
}

}  // namespace

cudaError_t launch_resident(const ScoreParams& p, int n_cols, int w_pad, int grid, cudaStream_t st) {
    if (n_cols == 32) {
        if (w_pad == 8) return launch_res<32, 8>(p, grid, st);
        if (w_pad == 16) return launch_res<32, 16>(p, grid, st);
        if (w_pad == 32) return launch_res<32, 32>(p, grid, st);
    } else if (n_cols == 64) {
        if (w_pad == 8) return launch_res<64, 8>(p, grid, st);
        if (w_pad == 16) return launch_res<64, 16>(p, grid, st);
        if (w_pad == 32) return launch_res<64, 32>(p, grid, st);
        if (w_pad == 64) return launch_res<64, 64>(p, grid, st);
    }
    return cudaErrorInvalidValue;
}

// The kernels that take the work-item tables of ScoreParams: the TMEM-resident two-pass kernel
// (above) and the single pass with the window rows' lse given (score_lse.cu).  One launch per
// slice of rounds whose items and units fit the parameter tables.
cudaError_t launch_score(const ScoreLaunch& L, cudaStream_t stream) {
    static_assert(sizeof(ScoreParams) <= 32000, "kernel parameters");
    static ScoreParams p;  // ~25 KB, kept off the host stack; calls are serialised by `mu`
    static std::mutex mu;
    std::lock_guard<std::mutex> lock(mu);
    memset(&p, 0, sizeof(p));
    p.tmap_k = L.tmap_k;
    p.tmap_q = L.tmap_q;
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
    p.wait_cycles = wait_limit_cycles();
    p.lse = L.lse;
    p.lse_stride = L.lse_head_stride;
    for (int b = 0; b < L.nb; ++b) {
        p.batch_group[b] = static_cast<int16_t>(L.batch_group[b]);
        p.batch_first[b] = static_cast<int16_t>(L.batch_first[b]);
        p.batch_nheads[b] = static_cast<int16_t>(L.batch_nheads[b]);
    }
    for (int i = 0; i < L.n_sel; ++i) p.sel_heads[i] = static_cast<int16_t>(L.sel_heads[i]);
    if (!L.lse && !L.resident) return cudaErrorInvalidValue;  // two-pass reload: score_layers.cu
    for (const ScoreSlice& sl : L.slices) {
        p.n_rounds = sl.n_rounds;
        p.n_items = sl.n_rounds * L.grid;
        p.n_units = sl.n_units;
        memcpy(p.items, L.items.data() + sl.item0, sizeof(ScoreItem) * p.n_items);
        memcpy(p.units, L.units.data() + sl.unit0, sizeof(ScoreUnit) * p.n_units);
        cudaError_t e = cudaSuccess;
        if (!L.lse) {  // the unit arrival counters of the exchange
            e = cudaMemsetAsync(L.counters, 0, sizeof(int) * sl.n_units, stream);
            if (e != cudaSuccess) return e;
        }
        e = L.lse ? launch_given_lse(p, L.n_cols, L.w_pad, L.grid, stream)
                  : launch_resident(p, L.n_cols, L.w_pad, L.grid, stream);
        if (e != cudaSuccess) return e;
    }
    return cudaSuccess;
}

}  // namespace ckv
