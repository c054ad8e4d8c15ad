// Window-attention scoring (arxiv 2508.02401, Sec. 3.3 with the attention of Eq. 2):
//
//   a_h[j] = sum_{r < w, j <= P+r} exp(s_{h,r,j} - lse_{h,r}),   s_{h,r,j} = scale * q_{h,r}.k_j
//
// for every selected head h of a KV group, every window row r and every key j of a sequence
// (P = L - w).  A row's normaliser lse needs every key before any probability can be summed
// over rows, so each key tile is used twice: once for the row statistics (pass 1), once for
// the probabilities (pass 2).
//
// Work: a unit is (sequence, batch of selected heads of one KV group); its key tiles are cut
// into items of a few tiles, and the items are dealt out in rounds of gridDim.x (CTA b takes
// item round * gridDim.x + b; all items of a unit are in one round).  One cooperative
// launch, one CTA per SM, 512 threads, warp-specialised:
//   warp 0       TMA producer for both passes, one polling thread: per item, TMA loads of the
//                window query rows (the MMA's B operand) into one of three buffers, then of its
//                128-key x 128-dim bf16 K tiles (two 128-byte-swizzled boxes of 64 dims) into
//                the pass-1 ring of kP1Slots slots; the same tiles again into the pass-2 ring
//                of kP2Slots slots once the item's pass-1 loads are out, so they come from L2;
//   warp 1       allocates TMEM and issues the pass-1 tcgen05.mma (M = 128 keys, N = the
//                window rows of a head batch, K = 128) into four pass-1 TMEM accumulators;
//   warp 2       issues the pass-2 tcgen05.mma into four pass-2 accumulators (two issuing
//                threads, so that neither pass's issue waits behind the other's);
//   warp 3       publisher and combiner: once an item's pass-1 partials are stored, one
//                release on the unit's arrival counter; then a bounded acquire spin until every
//                item of the unit has arrived and (for a unit of at most kWarpCombineMax items)
//                the combine of their partials into the unit's lse, left in shared memory for
//                pass 2 while pass 2 still works on the item before;
//   warps 4-11   pass 1, one warpgroup per 32 columns: each thread owns one key (one TMEM
//                lane) and keeps a running (max, sum of 2^(x - max)) per column; at the end of
//                the item the warpgroup's per-column partial goes to global memory;
//   warps 12-15  pass 2, one warpgroup over all N columns: takes the unit's lse from warp 3
//                (combining it itself, 128 threads, for a unit of more items) and sums
//                2^(x - lse) over each head's rows per key.
// Only the last tiles of a sequence (the window's own keys, the padding past its end) need a
// per-column mask; the others take an unmasked path of packed fp32 pair instructions.
// Pass 1 of an item overlaps the exchange and pass 2 of the item before it, so HBM keeps
// streaming while the CTAs wait for each other.
#include "score_common.cuh"

#include <string.h>

#include <mutex>

namespace ckv {

constexpr int kP1Slots = 3;                           // pass-1 ring (HBM)
constexpr int kP2Slots = 2;                           // pass-2 ring (L2)
constexpr int kAcc = 4;                               // TMEM accumulators per pass
constexpr int kQBufs = 3;                             // query-row buffers: pass 1 runs two items ahead
constexpr int kWarpCombineMax = 16;                   // units of more items: pass 2 combines (128 threads)

template <int N>
struct SmemLayout {
    static constexpr int kP1 = 0;
    static constexpr int kP2 = kP1 + kP1Slots * kTileBytes;
    static constexpr int kQ = kP2 + kP2Slots * kTileBytes;
    static constexpr int kQBytes = N * 256;             // one item's rows: N x 128 bf16
    static constexpr int kQHalf = N * 128;              // 64 dims of them
    static constexpr int kBars = kQ + kQBufs * kQBytes;
    // mbarrier indices, in this order
    static constexpr int kFull1 = 0, kFree1 = kFull1 + kP1Slots, kFull2 = kFree1 + kP1Slots,
                         kFree2 = kFull2 + kP2Slots, kAFull = kFree2 + kP2Slots,
                         kAEmpty = kAFull + kAcc, kBFull = kAEmpty + kAcc, kBEmpty = kBFull + kAcc,
                         kQFull = kBEmpty + kAcc, kQEmpty = kQFull + kQBufs,
                         kDone = kQEmpty + kQBufs, kGroup = kDone + 2,  // A0 A1 B
                         kPubFull = kGroup + 3, kPubEmpty = kPubFull + 2,
                         kLseFull = kPubEmpty + 2, kLseEmpty = kLseFull + 2,
                         kNumBars = kLseEmpty + 2;
    static constexpr int kTmemSlot = kBars + 8 * kNumBars;
    static constexpr int kAbort = kTmemSlot + 4;
    static constexpr int kBytes = kAbort + 4;
    static constexpr int kDynamic = kBytes + 1024;      // slack to align the base to 1024 B
};

// The unit's -lse per column (log2 units, -inf for a column without a real window row or
// without a visible key) from its items' partials, by one warp: lane 0 waits (bounded acquire
// spin) until every item of the unit has published, then, if `combine`, lane l combines the
// column pair (2l, 2l + 1) over the items, kU partials in flight (a unit of many items is
// combined by the pass-2 warpgroup instead, which has the threads for more loads in flight).
template <int N, int W_PAD>
__device__ __forceinline__ bool warp_unit_lse(const ScoreParams& p, const ScoreUnit& U, int unit,
                                              int lane, float* nlse, bool combine,
                                              volatile int* abort, long long lim) {
    constexpr int kNW = N / kCols, kPairs = N / 2, kU = 4;
    int got = 1;
    if (lane == 0) {
        const int target = U.nitems * kNW;
        const long long t0 = clock64();
        for (uint32_t k = 1; ld_acquire(p.counters + unit) < target; ++k) {
            __nanosleep(32);
            if ((k & 63u) == 0u && (*abort || clock64() - t0 > lim)) {
                got = 0;
                break;
            }
        }
    }
    __syncwarp();  // the acquire above orders the other lanes' reads of the partials too
    if (__shfl_sync(0xffffffffu, got, 0) == 0) return false;
    if (combine && lane < kPairs) {
        const float4* src = reinterpret_cast<const float4*>(p.partials + static_cast<size_t>(U.first_item) * N) + lane;
        float M0 = -INFINITY, S0 = 0.f, M1 = -INFINITY, S1 = 0.f;
        for (int k0 = 0; k0 < U.nitems; k0 += kU) {
            float4 pr[kU];
#pragma unroll
            for (int u = 0; u < kU; ++u)
                pr[u] = k0 + u < U.nitems ? __ldcg(src + static_cast<size_t>(k0 + u) * kPairs)
                                          : make_float4(-INFINITY, 0.f, -INFINITY, 0.f);
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
        const int nheads = p.batch_nheads[U.batch];
        const int c0 = 2 * lane, c1 = c0 + 1;
        const bool real0 = (c0 % W_PAD) < p.w && (c0 / W_PAD) < nheads;
        const bool real1 = (c1 % W_PAD) < p.w && (c1 / W_PAD) < nheads;
        nlse[c0] = real0 && S0 > 0.f ? -(M0 + lg2_approx(S0)) : -INFINITY;
        nlse[c1] = real1 && S1 > 0.f ? -(M1 + lg2_approx(S1)) : -INFINITY;
    }
    __syncwarp();
    return true;
}

template <int N, int W_PAD>
__global__ void __launch_bounds__(kThreads, 1) score_kernel(const __grid_constant__ ScoreParams p) {
    static_assert(N == 32 || N == 64, "N");
    static_assert(W_PAD == 8 || W_PAD == 16 || W_PAD == 32 || W_PAD == 64, "W_PAD");
    static_assert(W_PAD <= N, "a head's rows fit in one MMA");
    constexpr int kNW = N / kCols;                      // warpgroups per pass
    constexpr int kTmemCols = 2 * kAcc * N;           // pass-1 accumulators, then pass-2
    using SL = SmemLayout<N>;
    constexpr uint32_t kIdesc = idesc_bf16_f32(kTileKeys, N);

    extern __shared__ uint8_t smem_raw[];
    uint8_t* sm = reinterpret_cast<uint8_t*>(
        (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
    uint8_t* ring1 = sm + SL::kP1;
    uint8_t* ring2 = sm + SL::kP2;
    uint8_t* qbuf = sm + SL::kQ;
    uint64_t* bars = reinterpret_cast<uint64_t*>(sm + SL::kBars);
    uint64_t* full1 = bars + SL::kFull1;
    uint64_t* free1 = bars + SL::kFree1;
    uint64_t* full2 = bars + SL::kFull2;
    uint64_t* free2 = bars + SL::kFree2;
    uint64_t* a_full = bars + SL::kAFull;
    uint64_t* a_empty = bars + SL::kAEmpty;
    uint64_t* b_full = bars + SL::kBFull;
    uint64_t* b_empty = bars + SL::kBEmpty;
    uint64_t* q_full = bars + SL::kQFull;
    uint64_t* q_empty = bars + SL::kQEmpty;
    uint64_t* done = bars + SL::kDone;
    uint64_t* group = bars + SL::kGroup;        // one per epilogue warpgroup: A0 A1 B
    uint64_t* pub_full = bars + SL::kPubFull;   // pass-1 partials of an item stored (item parity)
    uint64_t* pub_empty = bars + SL::kPubEmpty;
    uint64_t* lse_full = bars + SL::kLseFull;   // a unit's lse is in nlse_s[item parity]
    uint64_t* lse_empty = bars + SL::kLseEmpty; // pass 2 is done with nlse_s[item parity]
    // scratch of the epilogues (static, so that its accesses are shared-memory instructions)
    __shared__ float2 red_a[2][2][128];  // [item parity][warpgroup][warp * 32 + lane]
    __shared__ __align__(16) float nlse_s[2][64];  // -lse per column, by item parity
    __shared__ float2 red_b[256];                     // pass-2 combine of a many-item unit
    uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(sm + SL::kTmemSlot);
    volatile int* abort = reinterpret_cast<volatile int*>(sm + SL::kAbort);

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;

    if (threadIdx.x == 0) {
        for (int i = 0; i < kP1Slots; ++i) {
            mbar_init(&full1[i], 1);
            mbar_init(&free1[i], 1);
        }
        for (int i = 0; i < kP2Slots; ++i) {
            mbar_init(&full2[i], 1);
            mbar_init(&free2[i], 1);
        }
        for (int i = 0; i < kAcc; ++i) {
            mbar_init(&a_full[i], 1);
            mbar_init(&a_empty[i], 4 * kNW);  // one arrival per pass-1 warp
            mbar_init(&b_full[i], 1);
            mbar_init(&b_empty[i], 4);        // one arrival per pass-2 warp
        }
        for (int i = 0; i < kQBufs; ++i) {
            mbar_init(&q_full[i], 1);
            mbar_init(&q_empty[i], 2);  // one commit per pass
        }
        mbar_init(&done[0], 1);
        mbar_init(&done[1], 1);
        for (int i = 0; i < 3; ++i) mbar_init(&group[i], kGroupArrivals);
        for (int i = 0; i < 2; ++i) {
            mbar_init(&pub_full[i], 32 * kNW);
            mbar_init(&pub_empty[i], 1);
            mbar_init(&lse_full[i], 1);
            mbar_init(&lse_empty[i], 4);  // one arrival per pass-2 warp
        }
        *abort = 0;
        fence_mbar_init();
        tma_prefetch_desc(&p.tmap_k);
        tma_prefetch_desc(&p.tmap_q);
    }
    // Query slots of head batches with fewer heads than the MMA's columns are never loaded;
    // zeros there keep those (unused) columns finite.
    for (int i = threadIdx.x; i < kQBufs * SL::kQBytes / 16; i += kThreads)
        reinterpret_cast<uint4*>(qbuf)[i] = make_uint4(0u, 0u, 0u, 0u);
    fence_proxy_async_smem();
    if (warp == 1) {
        tmem_alloc(tmem_slot, kTmemCols);
        tmem_relinquish();
    }
    if (blockIdx.x == 0 && threadIdx.x == 64 && seqlens_hash(p.cu_seqlens, p.S) != p.cu_hash)
        record_error(p.status, kDevBadSeqlens, 100);
    tc_fence_before_sync();
    __syncthreads();
    tc_fence_after_sync();
    const uint32_t tmem_base = *tmem_slot;
    // Registers: launched at 128 per thread (512 x 128 = 65536); on entry the producer/MMA/
    // query warpgroup gives up to 56, which leaves room for the two pass-1 warpgroups' 160;
    // the pass-2 warpgroup keeps 128 (128*56 + 256*160 + 128*128 = 64512).
    const int R = p.n_rounds;
    const int G = gridDim.x;
    // Limit of the waits on other roles and other CTAs (the waits for this block's own copies
    // and MMAs before it exits keep the long default, whatever this is).
    const long long lim = p.wait_cycles;
    auto item_of = [&](int r) -> const ScoreItem& { return p.items[r * G + blockIdx.x]; };

    if (warp < kWarpA) {
    setmaxnreg_dec<56>();
    if (warp == 0) {
        // ------------------------------------------------------------ TMA producer
        // Both rings from one thread that polls: a pass-1 slot still in use must not hold up
        // a pass-2 load, nor the other way round.
        if (lane == 0) {
            // Pass-1 tiles are read again by pass 2 shortly after: ask L2 to keep them, and to
            // drop them first once pass 2 has read them.
            const uint64_t pol1 = l2_policy_evict_last(), pol2 = l2_policy_evict_first();
            auto next_item = [&](int r) {
                while (r < R && item_of(r).ntiles == 0) ++r;
                return r;
            };
            int r1 = next_item(0), jt1 = 0, it1 = 0, use1 = 0;
            int r2 = r1, jt2 = 0, it2 = 0, use2 = 0;
            ScoreItem I1{}, I2{};
            ScoreUnit U1{}, U2{};
            if (r1 < R) {
                I1 = I2 = item_of(r1);
                U1 = U2 = p.units[I1.unit];
            }
            bool q_out = false, ok = true;
            long long t0 = clock64();
            uint32_t idle = 0;
            while (r1 < R || r2 < R) {
                bool did = false;
                if (r1 < R) {
                    if (!q_out) {
                        // The item's window query rows: per head of the batch two boxes of 64
                        // dims x W_PAD rows in the MMA's 128-byte-swizzled layout.  Rows past w
                        // (the next sequence's, or zeros past the end) and head slots past the
                        // batch's heads land in columns that the epilogues mask out.
                        const int qb = it1 % kQBufs;
                        if (mbar_test(&q_empty[qb], ((it1 / kQBufs) & 1) ^ 1)) {
                            uint8_t* qdst = qbuf + qb * SL::kQBytes;
                            const int first_row = p.batch_first[U1.batch], nheads = p.batch_nheads[U1.batch];
                            mbar_arrive_expect_tx(&q_full[qb], static_cast<uint32_t>(nheads * W_PAD * 256));
                            for (int slot = 0; slot < nheads; ++slot) {
                                const int h = p.sel_heads[first_row + slot];
                                uint8_t* d = qdst + slot * W_PAD * 128;
                                tma_load_3d(d, &p.tmap_q, &q_full[qb], 0, h, U1.seq * p.w);
                                tma_load_3d(d + SL::kQHalf, &p.tmap_q, &q_full[qb], 64, h, U1.seq * p.w);
                            }
                            q_out = true;
                            did = true;
                        }
                    }
                    const int s = use1 % kP1Slots;
                    if (q_out && mbar_test(&free1[s], ((use1 / kP1Slots) & 1) ^ 1)) {
                        mbar_arrive_expect_tx(&full1[s], kTileBytes);
                        uint8_t* dst = ring1 + s * kTileBytes;
                        const int g = p.batch_group[U1.batch];
                        const int tok = U1.seq_start + (I1.tile0 + jt1) * kTileKeys;
                        tma_load_3d_hint(dst, &p.tmap_k, &full1[s], 0, g, tok, pol1);
                        tma_load_3d_hint(dst + kHalfBytes, &p.tmap_k, &full1[s], 64, g, tok, pol1);
                        ++use1;
                        did = true;
                        if (++jt1 == I1.ntiles) {
                            jt1 = 0;
                            ++it1;
                            q_out = false;
                            r1 = next_item(r1 + 1);
                            if (r1 < R) {
                                I1 = item_of(r1);
                                U1 = p.units[I1.unit];
                            }
                        }
                    }
                }
                // pass 2 of an item follows its pass-1 loads, so that it reads L2
                if (r2 < R && it2 < it1) {
                    const int s = use2 % kP2Slots;
                    if (mbar_test(&free2[s], ((use2 / kP2Slots) & 1) ^ 1)) {
                        mbar_arrive_expect_tx(&full2[s], kTileBytes);
                        uint8_t* dst = ring2 + s * kTileBytes;
                        const int g = p.batch_group[U2.batch];
                        const int tok = U2.seq_start + (I2.tile0 + jt2) * kTileKeys;
                        tma_load_3d_hint(dst, &p.tmap_k, &full2[s], 0, g, tok, pol2);
                        tma_load_3d_hint(dst + kHalfBytes, &p.tmap_k, &full2[s], 64, g, tok, pol2);
                        ++use2;
                        did = true;
                        if (++jt2 == I2.ntiles) {
                            jt2 = 0;
                            ++it2;
                            r2 = next_item(r2 + 1);
                            if (r2 < R) {
                                I2 = item_of(r2);
                                U2 = p.units[I2.unit];
                            }
                        }
                    }
                }
                if (did) {
                    idle = 0;
                    t0 = clock64();
                } else {
                    __nanosleep(32u << (idle < 1u ? idle : 1u));
                    if ((++idle & 15u) == 0u && (*abort || clock64() - t0 > lim)) {
                        ok = false;
                        break;
                    }
                }
            }
            if (!ok) {
                *abort = 1;
                record_error(p.status, kDevTimeout, 10);
            }
            // Let every issued copy land before the block may exit.
            volatile int never = 0;
            for (int k = (use1 > kP1Slots ? use1 - kP1Slots : 0); k < use1; ++k)
                mbar_wait(&full1[k % kP1Slots], (k / kP1Slots) & 1, &never);
            for (int k = (use2 > kP2Slots ? use2 - kP2Slots : 0); k < use2; ++k)
                mbar_wait(&full2[k % kP2Slots], (k / kP2Slots) & 1, &never);
            const int nq = it1 + (q_out ? 1 : 0);
            for (int k = (nq > kQBufs ? nq - kQBufs : 0); k < nq; ++k)
                mbar_wait(&q_full[k % kQBufs], (k / kQBufs) & 1, &never);
        }
    } else if (warp == 1 || warp == 2) {
        // ------------------------------------------------------------ MMA issuers
        // warp 1: pass 1, warp 2: pass 2, so that neither pass's issue waits behind the other's.
        if (lane == 0) {
            const bool first = warp == 1;
            const int nslots = first ? kP1Slots : kP2Slots;
            const uint8_t* ring = first ? ring1 : ring2;
            uint64_t* full = first ? full1 : full2;
            uint64_t* freed = first ? free1 : free2;
            uint64_t* acc_full = first ? a_full : b_full;
            uint64_t* acc_empty = first ? a_empty : b_empty;
            uint64_t* fin = first ? done : done + 1;
            const uint32_t d0 = tmem_base + static_cast<uint32_t>((first ? 0 : kAcc) * N);
            int it = 0, use = 0;
            bool ok = true;
            for (int r = 0; ok && r < R; ++r) {
                const int n = item_of(r).ntiles;
                if (n == 0) continue;
                const int qb = it % kQBufs;
                if (!mbar_wait(&q_full[qb], (it / kQBufs) & 1, abort, lim)) {
                    ok = false;
                    break;
                }
                const uint32_t b0 = smem_u32(qbuf + qb * SL::kQBytes);
                for (int jt = 0; jt < n; ++jt, ++use) {
                    const int s = use % nslots, acc = use % kAcc;
                    if (!mbar_wait(&full[s], (use / nslots) & 1, abort, lim) ||
                        !mbar_wait(&acc_empty[acc], ((use / kAcc) & 1) ^ 1, abort, lim)) {
                        ok = false;
                        break;
                    }
                    tc_fence_after_sync();
                    const uint32_t a0 = smem_u32(ring + s * kTileBytes);
                    const uint32_t d = d0 + static_cast<uint32_t>(acc * N);
#pragma unroll
                    for (int kk = 0; kk < kHeadDim / 16; ++kk) {
                        const uint32_t koff = (kk & 3) * 32;
                        const uint64_t ad = sdesc_k_major_sw128(a0 + (kk >> 2) * kHalfBytes + koff);
                        const uint64_t bd = sdesc_k_major_sw128(b0 + (kk >> 2) * SL::kQHalf + koff);
                        umma_bf16(d, ad, bd, kIdesc, kk > 0 ? 1u : 0u);
                    }
                    umma_commit(&acc_full[acc]);
                    umma_commit(&freed[s]);
                }
                if (!ok) break;
                umma_commit(&q_empty[qb]);  // this pass is done with the item's query rows
                ++it;
            }
            if (!ok) {
                *abort = 1;
                record_error(p.status, kDevTimeout, first ? 11 : 12);
            }
            umma_commit(fin);
            volatile int never = 0;
            mbar_wait(fin, 0, &never);
        }
        __syncwarp();
    } else if (warp == 3) {
        // ------------------------------------------------------------ publisher and combiner
        // Per item: once both pass-1 warpgroups have stored its partials (their pub_full
        // arrival releases them to lane 0 at CTA scope), one release add on the unit's arrival
        // counter makes them visible GPU-wide (a release is cumulative).  Then the warp waits
        // for the unit's other items, combines all their partials into the unit's lse and
        // leaves it in nlse_s for pass 2, which meanwhile still works on the item before: the
        // exchange stays off pass 2's path unless pass 1 elsewhere is late.
        int it = 0;
        bool ok = true;
        for (int r = 0; r < R; ++r) {
            const ScoreItem I = item_of(r);
            if (I.ntiles == 0) continue;
            const int buf = it & 1;
            int good = 1;
            if (lane == 0) {
                if (!mbar_wait(&pub_full[buf], (it >> 1) & 1, abort, lim)) {
                    good = 0;
                } else {
                    red_release_add(p.counters + I.unit, kNW);
                    mbar_arrive(&pub_empty[buf]);
                    good = mbar_wait(&lse_empty[buf], ((it >> 1) & 1) ^ 1, abort, lim) ? 1 : 0;
                }
            }
            const ScoreUnit& U = p.units[I.unit];
            if (__shfl_sync(0xffffffffu, good, 0) == 0 ||
                !warp_unit_lse<N, W_PAD>(p, U, I.unit, lane, nlse_s[buf], U.nitems <= kWarpCombineMax,
                                         abort, lim)) {
                ok = false;
                break;
            }
            if (lane == 0) mbar_arrive(&lse_full[buf]);
            ++it;
        }
        if (!ok && lane == 0) {
            *abort = 1;
            record_error(p.status, kDevTimeout, 17);
        }
    }
    } else if (warp < kWarpB) {
        // ------------------------------------------------------------ pass 1
        setmaxnreg_inc<160>();
        const int wg = (warp - kWarpA) >> 2;  // columns [wg*32, wg*32+32)
        if (wg < kNW) {
            const int eq = warp & 3;            // TMEM lane quarter
            const int wtid = threadIdx.x - (kWarpA + 4 * wg) * 32;  // 0 .. 127
            const int col0 = wg * kCols;
            const uint32_t lane_base = static_cast<uint32_t>(eq * 32) << 16;
            uint64_t* gbar = &group[wg];
            uint32_t gphase = 0;
            int a_it = 0, a_item = 0;
            bool ok = true;
            for (int r = 0; ok && r < R; ++r) {
                const int item = r * G + blockIdx.x;
                const ScoreItem I = p.items[item];
                const int n = I.ntiles;
                if (n == 0) continue;
                const ScoreUnit U = p.units[I.unit];
                const int L = U.len, P = L - p.w;
                const float sl2 = p.sl2;
                // Running maximum (log2 units, kept negated so that it is the FMA's addend) and
                // the sum relative to it.  -1e30 (not -inf) for a column with no visible key
                // yet keeps the reductions below free of inf - inf.
                float nm[kCols], sm_[kCols];
#pragma unroll
                for (int i = 0; i < kCols; ++i) {
                    nm[i] = 1e30f;
                    sm_[i] = 0.f;
                }
                for (int jt = 0; jt < n; ++jt, ++a_it) {
                    const int acc = a_it % kAcc;
                    if (!mbar_wait(&a_full[acc], (a_it / kAcc) & 1, abort, lim)) {
                        ok = false;
                        break;
                    }
                    tc_fence_after_sync();
                    const int t = I.tile0 + jt;
                    const int j = t * kTileKeys + eq * 32 + lane;  // sequence-local key
                    // Tiles wholly before the window, inside the sequence: every key is seen by
                    // every row, and the columns without a real row are never read, so no mask.
                    const bool edge = (t * kTileKeys + kTileKeys - 1 >= P) || (t * kTileKeys + kTileKeys > L);
                    const uint32_t taddr = tmem_base + lane_base + static_cast<uint32_t>(acc * N + col0);
                    // both halves of 16 columns in flight, then one wait
                    float vv[2][16];
                    tmem_ld16_nowait(taddr, vv[0]);
                    tmem_ld16_nowait(taddr + 16, vv[1]);
                    tmem_ld_wait();
                    reg_fence(vv[0]);
                    reg_fence(vv[1]);
                    tc_fence_before_sync();
                    __syncwarp();
                    if (lane == 0) mbar_arrive(&a_empty[acc]);  // the accumulator is free
                    if (!edge) {
                        stats_block<false, W_PAD, 0>(vv[0], nm, sm_, sl2, 0);
                        stats_block<false, W_PAD, 16>(vv[1], nm + 16, sm_ + 16, sl2, 0);
                    } else {
                        // row r of a head sees key j iff r >= j - P; keys past L are padding
                        // (columns without a real row are never read, so they need no mask)
                        const int jr = (j < L ? j - P : (1 << 30)) - (W_PAD == 64 ? col0 : 0);
                        stats_block<true, W_PAD, 0>(vv[0], nm, sm_, sl2, jr);
                        stats_block<true, W_PAD, 16>(vv[1], nm + 16, sm_ + 16, sl2, jr);
                    }
                }
                float m[kCols];
#pragma unroll
                for (int i = 0; i < kCols; ++i) m[i] = -nm[i];
                if (!ok) break;
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
                record_error(p.status, kDevTimeout, 14);
            }
        }
    } else {
        // ------------------------------------------------------------ pass 2
        // One warpgroup over all N columns; lse sits in shared memory and is read by every
        // lane of a warp at the same address.
        const int eq = warp & 3;
        const int wtid = threadIdx.x - kWarpB * 32;  // 0 .. 127
        const uint32_t lane_base = static_cast<uint32_t>(eq * 32) << 16;
        uint64_t* gbar = &group[2];
        uint32_t gphase = 0;
        constexpr int kHeads = N / W_PAD;  // head slots of the MMA's columns
        int b_it = 0, n_item = 0;
        bool ok = true;
        for (int r = 0; ok && r < R; ++r) {
            const ScoreItem I = p.items[r * G + blockIdx.x];
            const int n = I.ntiles;
            if (n == 0) continue;
            const ScoreUnit U = p.units[I.unit];
            const int L = U.len, P = L - p.w;
            const int first = p.batch_first[U.batch], nheads = p.batch_nheads[U.batch];
            const int T = p.T;
            const float sl2 = p.sl2;
            float* const scores = p.scores;
            // ---------------------------------------------------- the unit's lse (warp 3)
            const int buf = n_item & 1;
            int good = 1;
            if (lane == 0) good = mbar_wait(&lse_full[buf], (n_item >> 1) & 1, abort, lim) ? 1 : 0;
            __syncwarp();
            if (__shfl_sync(0xffffffffu, good, 0) == 0) {
                ok = false;
                break;
            }
            if (U.nitems > kWarpCombineMax) {  // warp 3 only acquired: combine here
                uint64_t colmask = 0;           // columns that hold a real window row
#pragma unroll
                for (int c = 0; c < N; ++c)
                    if ((c % W_PAD) < p.w && (c / W_PAD) < nheads) colmask |= 1ull << c;
                if (!unit_combine<N>(p, U, wtid, gbar, gphase, red_b, nlse_s[buf], colmask, abort, lim)) {
                    ok = false;
                    break;
                }
            }
            const float* nlse = nlse_s[buf];
            // ---------------------------------------------------- the item's tiles
            for (int jt = 0; jt < n; ++jt, ++b_it) {
                const int acc = b_it % kAcc;
                if (!mbar_wait(&b_full[acc], (b_it / kAcc) & 1, abort, lim)) {
                    ok = false;
                    break;
                }
                tc_fence_after_sync();
                const int t = I.tile0 + jt;
                const int j = t * kTileKeys + eq * 32 + lane;
                const bool edge = (t * kTileKeys + kTileKeys - 1 >= P) || (t * kTileKeys + kTileKeys > L);
                const uint32_t taddr = tmem_base + lane_base + static_cast<uint32_t>((kAcc + acc) * N);
                // every 16-column chunk in flight, then one wait
                float vv[N / 16][16];
#pragma unroll
                for (int hh = 0; hh < N / 16; ++hh) tmem_ld16_nowait(taddr + hh * 16, vv[hh]);
                tmem_ld_wait();
#pragma unroll
                for (int hh = 0; hh < N / 16; ++hh) reg_fence(vv[hh]);
                tc_fence_before_sync();
                __syncwarp();
                if (lane == 0) mbar_arrive(&b_empty[acc]);  // the accumulator is free
                float accum[kHeads];
                if (!edge) {
                    prob_sums<N, W_PAD, false>(vv, sl2, nlse, 0, accum);
                } else {  // row r sees key j iff r >= j - P; keys past L are padding
                    prob_sums<N, W_PAD, true>(vv, sl2, nlse, j < L ? j - P : (1 << 30), accum);
                }
                if (j < L) {
                    const size_t col = static_cast<size_t>(U.seq_start) + j;
#pragma unroll
                    for (int h = 0; h < kHeads; ++h)
                        if (h < nheads) scores[static_cast<size_t>(first + h) * T + col] = accum[h];
                }
            }
            __syncwarp();
            if (lane == 0) mbar_arrive(&lse_empty[buf]);  // this warp is done with the lse
            ++n_item;
        }
        if (!ok) {
            *abort = 1;
            record_error(p.status, kDevTimeout, 16);
        }
    }

    tc_fence_before_sync();
    __syncthreads();
    if (warp == 1) {
        tc_fence_after_sync();
        tmem_dealloc(tmem_base, kTmemCols);
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
    // One launch per slice of rounds whose items and units fit the parameter tables.
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
            : L.resident ? launch_resident(p, L.n_cols, L.w_pad, L.grid, stream)
                         : dispatch(p, L.n_cols, L.w_pad, L.grid, stream);
        if (e != cudaSuccess) return e;
    }
    return cudaSuccess;
}

}  // namespace ckv
