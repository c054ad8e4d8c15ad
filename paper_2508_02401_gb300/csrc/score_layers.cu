// Window-attention scoring of several layers in one persistent launch (arxiv 2508.02401,
// Sec. 3.3 with the attention of Eq. 2):
//
//   a_h[j] = sum_{r < w, j <= P+r} exp(s_{h,r,j} - lse_{h,r}),   s_{h,r,j} = scale * q_{h,r}.k_j
//
// for every selected head h of every KV group of every layer of the launch, every window row r
// and every key j of a sequence (P = L - w).  A row's normaliser lse needs every key before any
// probability can be summed over rows, so each key tile is used twice: once for the row
// statistics (pass 1, from HBM), once for the probabilities (pass 2, from L2).
//
// Work: a unit is (layer, head batch of one KV group, sequence); its key tiles are split into
// m items of balanced length, m at most the CTAs of the launch.  The items of all units, unit
// after unit, form one sequence; the CTAs take them dynamically, one at a time, from a global
// counter, as each CTA becomes ready to start one (its query buffer is free).  The SMs do not
// stream HBM equally fast, and taking items on demand lets the faster ones take more, so that
// a unit's items finish close together and pass 2 re-reads its tiles while they are still in
// L2.  No wait can close a cycle: a CTA waits only for units it holds an item of, a unit's
// items are taken before any later unit's, and a CTA takes an item only when it can run its
// pass 1 (up to two items ahead of its pass 2); if a unit's items were all held by CTAs that
// cannot start them, each would hold three of the unit's items, more than the G it has.
//
// Exchange: at the end of an item, pass 1 leaves, per window-row column, its keys' sum
// sum_j 2^(x_j) (x = logit * log2 e) as (m, s) with the item's maximum m in shared memory; a
// publisher warp adds each s * 2^m in fp64 to the unit's accumulator with one atomic add and
// counts the item's arrival on the unit's counter with a release (the wait for its adds to
// land stays off pass 1's path).  A unit's lse per column is log2 of its accumulator once the
// counter is complete: one read of N doubles, whatever the number of items.  fp64 holds
// 2^(+-1022), so a column's largest logit times log2 e must lie within +-990 (about +-686 in
// natural log units); beyond that the status word reports kDevRange.
//
// One cooperative launch, one CTA per SM, 512 threads, warp-specialised:
//   warp 0       the producer, one polling thread: takes the CTA's next item from the global
//                counter and posts it to the other roles (a ring of item indices in shared
//                memory); per item, TMA loads of the window query rows into one of kQBufs
//                buffers, then of its 128-key x 128-dim bf16 K tiles (two 128-byte-swizzled
//                boxes of 64 dims) into the pass-1 ring (evict-last: pass 2 reads them again;
//                evict-first for the first fifth of an item of a long unit, whose re-reads
//                come too late for L2); the same tiles again into the pass-2 ring
//                (evict-first) once the item's pass-1 loads are out;
//   warp 1       allocates TMEM and issues the pass-1 tcgen05.mma (M = 128 keys, N = the
//                window rows of a head batch, K = 128) into four pass-1 accumulators;
//   warp 2       issues the pass-2 tcgen05.mma into four pass-2 accumulators;
//   warp 3       the publisher: per item, the fp64 atomic adds of its column sums and the
//                release of its arrival on the unit's counter;
//   warps 4-11   pass 1, one warpgroup per 32 columns: each thread owns one key (one TMEM
//                lane) and keeps a running (max, sum of 2^(x - max)) per column;
//   warps 12-15  pass 2, one warpgroup over all N columns: per item, a bounded acquire spin
//                until the item's unit is complete and the unit's -lse per column from its
//                accumulator, then per key the sums of 2^(x - lse) over each head's rows.
// Only the last tiles of a sequence (the window's own keys, the padding past its end) need a
// per-column mask; the others take an unmasked path of packed fp32 pair instructions.
#include "score_layers.cuh"

#include <string.h>

#include <mutex>

namespace ckv {

namespace {

constexpr int kP1Slots = 2;   // pass-1 ring (HBM)
constexpr int kP2Slots = 3;   // pass-2 ring (L2): pass 2 must outrun pass 1 after each exchange wait
constexpr int kAcc = 4;       // TMEM accumulators per pass
constexpr int kQBufs = 3;     // query-row buffers: pass 1 runs up to two items ahead of pass 2
// Units of more keys than this (16 MB of K, an eighth of L2) load the first fifth of each item's
// tiles evict-first in pass 1: their re-reads come after most of L2 has turned over.
constexpr int kLongUnitKeys = 65536;
constexpr int kItemRing = 8;  // item indices posted by the producer (more than any role's lag)
// Largest |log2| of an item's column maximum: an item's sum is then below 2^1000 (at most
// 2^10 keys), and the sum of up to 2^20 items stays below fp64's 2^1024.
constexpr double kMaxLog2 = 990.0;

template <int N>
struct LayersSmem {
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
                         kItemFull = kPubEmpty + 2, kItemFree = kItemFull + kItemRing,
                         kNumBars = kItemFree + kItemRing;
    static constexpr int kItems = kBars + 8 * kNumBars;  // int[kItemRing]: posted item indices
    static constexpr int kTmemSlot = kItems + 4 * kItemRing;
    static constexpr int kAbort = kTmemSlot + 4;
    static constexpr int kBytes = kAbort + 4;
    static constexpr int kDynamic = kBytes + 1024;      // slack to align the base to 1024 B
};
// dynamic + the kernel's static shared memory (under 6 KB) within the 227 KB a block may use
static_assert(LayersSmem<64>::kDynamic + 6 * 1024 <= 232448, "shared memory, N = 64");

// End of a pass-1 item for one warpgroup of kCols columns: per column, the warp maximum by
// redux and the sums rescaled to it, the warps' sums by recursive halving, then the four warps
// through shared memory `red`; thread c < kCols (the warpgroup's first warp) leaves column c's
// (max, sum) in `out[c]` once the publisher is done with that buffer's previous item, and
// arrives on pub_full.
__device__ __forceinline__ bool item_sums(float (&m)[kCols], float (&s)[kCols], float2* red, int eq,
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

// s * 2^M as a double, for |M| <= kMaxLog2: the power of two of floor(M) exactly (built from
// the exponent bits), the rest in fp32.
__device__ __forceinline__ double scaled_sum(float M, float S) {
    const float e = floorf(M);
    const double p2 = __longlong_as_double(static_cast<long long>(static_cast<int>(e) + 1023) << 52);
    return static_cast<double>(S * ex2_approx(M - e)) * p2;
}

template <int N, int W_PAD>
__global__ void __launch_bounds__(kThreads, 1) score_layers_kernel(const __grid_constant__ LayersParams p) {
    static_assert(N == 32 || N == 64, "N");
    static_assert(W_PAD == 8 || W_PAD == 16 || W_PAD == 32 || W_PAD == 64, "W_PAD");
    static_assert(W_PAD <= N, "a head's rows fit in one MMA");
    constexpr int kNW = N / kCols;                      // warpgroups per pass
    constexpr int kTmemCols = 2 * kAcc * N;             // pass-1 accumulators, then pass-2
    using SL = LayersSmem<N>;
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
    uint64_t* pub_full = bars + SL::kPubFull;   // pass 1 left an item's sums in pub_s[item parity]
    uint64_t* pub_empty = bars + SL::kPubEmpty; // the publisher is done with pub_s[item parity]
    uint64_t* item_full = bars + SL::kItemFull; // items[k] holds the CTA's next item index
    uint64_t* item_free = bars + SL::kItemFree; // every role has read items[k]
    int* items = reinterpret_cast<int*>(sm + SL::kItems);
    // scratch of the epilogues (static, so that its accesses are shared-memory instructions)
    __shared__ float2 red_a[2][2][128];  // [item parity][warpgroup][warp * 32 + lane]
    __shared__ float2 pub_s[2][64];      // [item parity][column]: (max, sum) of an item
    __shared__ __align__(16) float nlse_s[64];  // -lse per column of pass 2's item
    uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(sm + SL::kTmemSlot);
    volatile int* abort = reinterpret_cast<volatile int*>(sm + SL::kAbort);

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int n_items = p.n_items;

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
            mbar_init(&pub_full[i], 32 * kNW);  // the columns' threads of each pass-1 warpgroup
            mbar_init(&pub_empty[i], 1);
        }
        for (int i = 0; i < kItemRing; ++i) {
            mbar_init(&item_full[i], 1);
            mbar_init(&item_free[i], 4);  // one arrival per pass-2 warp, once it has read the entry
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
    for (int i = threadIdx.x; i < kQBufs * SL::kQBytes / 16; i += kThreads)
        reinterpret_cast<uint4*>(qbuf)[i] = make_uint4(0u, 0u, 0u, 0u);
    fence_proxy_async_smem();
    if (warp == 1) {
        tmem_alloc(tmem_slot, kTmemCols);
        tmem_relinquish();
    }
    if (blockIdx.x == 0 && threadIdx.x == 64 && seqlens_hash(p.cu_seqlens, p.S_all) != p.cu_hash)
        record_error(p.status, kDevBadSeqlens, 100);
    tc_fence_before_sync();
    __syncthreads();
    tc_fence_after_sync();
    const uint32_t tmem_base = *tmem_slot;
    // Registers: launched at 128 per thread (512 x 128 = 65536); on entry the producer/MMA/
    // lse warpgroup gives up to 56, which leaves room for the two pass-1 warpgroups' 160;
    // the pass-2 warpgroup keeps 128 (128*56 + 256*160 + 128*128 = 64512).
    // Limit of the waits on other roles and other CTAs (the waits for this block's own copies
    // and MMAs before it exits keep the long default, whatever this is).
    const long long lim = p.wait_cycles;

    if (warp < kWarpA) {
    setmaxnreg_dec<56>();
    if (warp == 0) {
        // ------------------------------------------------------------ producer
        // Items, and the tiles of both passes, from one thread that polls: a pass-1 slot still
        // in use must not hold up a pass-2 load, nor the other way round.
        if (lane == 0) {
            // Pass-1 tiles are read again by pass 2 shortly after: ask L2 to keep them, and to
            // drop them first once pass 2 has read them.
            const uint64_t pol1 = l2_policy_evict_last(), pol2 = l2_policy_evict_first();
            int* next_item = p.counters + p.n_units;
            // The window query rows of an item into query buffer qb (completion on q_full[qb]):
            // per head of the batch two boxes of 64 dims x W_PAD rows in the MMA's
            // 128-byte-swizzled layout.  Rows past w (the next sequence's, or zeros past the
            // end) and head slots past the batch's heads land in columns that the epilogues
            // mask out.
            auto load_q = [&](const Item& I, int qb) {
                uint8_t* qdst = qbuf + qb * SL::kQBytes;
                const int nheads = p.batch_nheads[I.batch], sel0 = p.batch_sel[I.batch];
                const CUtensorMap* qm = &p.tmap_q[I.layer];
                mbar_arrive_expect_tx(&q_full[qb], static_cast<uint32_t>(nheads * W_PAD * 256));
                const int row = (p.seq0 + I.seq) * p.w;
                for (int slot = 0; slot < nheads; ++slot) {
                    const int h = p.sel_heads[sel0 + slot];
                    uint8_t* d = qdst + slot * W_PAD * 128;
                    tma_load_3d(d, qm, &q_full[qb], 0, h, row);
                    tma_load_3d(d + SL::kQHalf, qm, &q_full[qb], 64, h, row);
                }
            };
            // it1: items taken (pass-1 cursor on the last one); it2: pass-2 cursor
            int it1 = 0, jt1 = 0, use1 = 0, it2 = 0, jt2 = 0, use2 = 0, have2 = -1;
            Item I1{}, I2{};
            bool have1 = false, ended = false, ok = true;
            long long t0 = clock64();
            uint32_t idle = 0;
            while (true) {
                bool did = false;
                if (!have1 && !ended) {
                    // Take the next item once its query buffer and its ring entry are free.
                    const int qb = it1 % kQBufs, k = it1 % kItemRing;
                    if (mbar_test(&q_empty[qb], ((it1 / kQBufs) & 1) ^ 1) &&
                        mbar_test(&item_free[k], ((it1 / kItemRing) & 1) ^ 1)) {
                        const int gi = atomicAdd(next_item, 1);
                        items[k] = gi < n_items ? gi : -1;
                        mbar_arrive(&item_full[k]);  // releases items[k] to the other roles
                        if (gi >= n_items) {
                            ended = true;
                        } else {
                            I1 = get_item(p, gi);
                            load_q(I1, qb);
                            have1 = true;
                            jt1 = 0;
                        }
                        did = true;
                    }
                }
                if (have1) {
                    const int s = use1 % kP1Slots;
                    if (mbar_test(&free1[s], ((use1 / kP1Slots) & 1) ^ 1)) {
                        mbar_arrive_expect_tx(&full1[s], kTileBytes);
                        uint8_t* dst = ring1 + s * kTileBytes;
                        const int g = p.batch_group[I1.batch];
                        const int tok = I1.start + (I1.tile0 + jt1) * kTileKeys;
                        const CUtensorMap* km = &p.tmap_k[I1.layer];
                        // In a long unit pass 2 re-reads an item's first tiles too late for L2
                        // anyway: loading them evict-first leaves L2 to the rest.
                        const uint64_t polx = (I1.len > kLongUnitKeys && jt1 * 5 < I1.ntiles) ? pol2 : pol1;
                        tma_load_3d_hint(dst, km, &full1[s], 0, g, tok, polx);
                        tma_load_3d_hint(dst + kHalfBytes, km, &full1[s], 64, g, tok, polx);
                        ++use1;
                        did = true;
                        if (++jt1 == I1.ntiles) {
                            have1 = false;
                            ++it1;
                        }
                    }
                }
                // pass 2 of an item follows its pass-1 loads, so that it reads L2
                if (it2 < it1) {
                    if (have2 != it2) {
                        I2 = get_item(p, items[it2 % kItemRing]);
                        have2 = it2;
                    }
                    const int s = use2 % kP2Slots;
                    if (mbar_test(&free2[s], ((use2 / kP2Slots) & 1) ^ 1)) {
                        mbar_arrive_expect_tx(&full2[s], kTileBytes);
                        uint8_t* dst = ring2 + s * kTileBytes;
                        const int g = p.batch_group[I2.batch];
                        const int tok = I2.start + (I2.tile0 + jt2) * kTileKeys;
                        const CUtensorMap* km = &p.tmap_k[I2.layer];
                        tma_load_3d_hint(dst, km, &full2[s], 0, g, tok, pol2);
                        tma_load_3d_hint(dst + kHalfBytes, km, &full2[s], 64, g, tok, pol2);
                        ++use2;
                        did = true;
                        if (++jt2 == I2.ntiles) {
                            jt2 = 0;
                            ++it2;
                        }
                    }
                }
                if (ended && !have1 && it2 == it1) break;
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
            const int nq = it1 + (have1 ? 1 : 0);
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
            int use = 0;
            bool ok = true;
            for (int it = 0; ok; ++it) {
                int gi = -1;
                if (!wait_item<kItemRing>(item_full, items, it, &gi, abort, lim)) {
                    ok = false;
                    break;
                }
                if (gi < 0) break;
                const int n = get_item(p, gi).ntiles;
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
        // ------------------------------------------------------------ publisher
        // Per item: once both pass-1 warpgroups have left its column sums (pub_full), lane l
        // adds columns l and l + 32 to the unit's fp64 accumulator, and lane 0 releases the
        // item's arrival on the unit's counter after a warp barrier.
        bool ok = true;
        for (int it = 0;; ++it) {
            int gi = -1, good = 1;
            if (lane == 0) good = wait_item<kItemRing>(item_full, items, it, &gi, abort, lim) ? 1 : 0;
            gi = __shfl_sync(0xffffffffu, gi, 0);
            if (__shfl_sync(0xffffffffu, good, 0) == 0) {
                ok = false;
                break;
            }
            if (gi < 0) break;
            const Item I = get_item(p, gi);
            const int buf = it & 1;
            if (lane == 0) good = mbar_wait(&pub_full[buf], (it >> 1) & 1, abort, lim) ? 1 : 0;
            if (__shfl_sync(0xffffffffu, good, 0) == 0) {
                ok = false;
                break;
            }
            double* dst = p.sums + static_cast<size_t>(I.unit) * N;
#pragma unroll
            for (int c = lane; c < N; c += 32) {
                const float2 ms = pub_s[buf][c];
                if (ms.y > 0.f) {
                    if (!(fabsf(ms.x) <= static_cast<float>(kMaxLog2))) record_error(p.status, kDevRange, c);
                    else atomicAdd(dst + c, scaled_sum(ms.x, ms.y));
                }
            }
            // the warp barrier orders every lane's adds before lane 0's release, and a release
            // is cumulative: a thread that acquires the count sees the adds of every item counted
            __syncwarp();
            if (lane == 0) {
                red_release_add(p.counters + I.unit, 1);
                mbar_arrive(&pub_empty[buf]);
            }
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
            int a_it = 0;
            bool ok = true;
            for (int it = 0; ok; ++it) {
                int gi = -1;
                if (!wait_item<kItemRing>(item_full, items, it, &gi, abort, lim)) {
                    ok = false;
                    break;
                }
                if (gi < 0) break;
                const Item I = get_item(p, gi);
                const int n = I.ntiles;
                const int L = I.len, P = L - p.w;
                const float sl2 = p.sl2;
                // Running maximum (log2 units, kept negated so that it is the FMA's addend) and
                // the sum relative to it.  -1e30 (not -inf) for a column with no visible key
                // yet keeps the reductions below free of inf - inf.
                float nm[kCols], sm_[kCols];
#pragma unroll
                for (int c = 0; c < kCols; ++c) {
                    nm[c] = 1e30f;
                    sm_[c] = 0.f;
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
                    float vv[2][16];  // both halves of 16 columns in flight, then one wait
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
                for (int c = 0; c < kCols; ++c) m[c] = -nm[c];
                if (!ok) break;
                if (!item_sums(m, sm_, red_a[it & 1][wg], eq, lane, wtid, gbar, gphase,
                               &pub_full[it & 1], &pub_empty[it & 1], (it >> 1) & 1,
                               pub_s[it & 1] + col0, abort, lim)) {
                    ok = false;
                    break;
                }
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
        constexpr int kHeads = N / W_PAD;  // head slots of the MMA's columns
        uint32_t gphase = 0;
        int b_it = 0;
        bool ok = true;
        for (int it = 0; ok; ++it) {
            int gi = -1, good = 1;
            if (lane == 0) good = wait_item<kItemRing>(item_full, items, it, &gi, abort, lim) ? 1 : 0;
            gi = __shfl_sync(0xffffffffu, gi, 0);
            if (__shfl_sync(0xffffffffu, good, 0) == 0) {
                ok = false;
                break;
            }
            if (gi < 0) break;
            // pass 2 reads an item's ring entry last: once each of its warps has, the producer
            // may post another item there
            if (lane == 0) mbar_arrive(&item_free[it % kItemRing]);
            const Item I = get_item(p, gi);
            const int n = I.ntiles, tile0 = I.tile0;
            const int L = I.len, P = L - p.w;
            const int nheads = p.batch_nheads[I.batch];
            const size_t T = static_cast<size_t>(p.T);
            const float sl2 = p.sl2;
            // the batch's first score row, at the sequence's first token
            float* const out = p.scores[I.layer] + static_cast<size_t>(p.batch_first[I.batch]) * T + I.start;
            // ---------------------------------------------------- the unit's lse
            // a bounded acquire spin until every item of the unit has arrived, carried to the
            // warpgroup by its barrier; then -lse per column from the accumulator
            if (threadIdx.x == kWarpB * 32) {
                const long long t0 = clock64();
                for (uint32_t k = 1; ld_acquire(p.counters + I.unit) < I.nitems; ++k) {
                    __nanosleep(32);
                    if ((k & 63u) == 0u && (*abort || clock64() - t0 > lim)) {
                        *abort = 1;
                        break;
                    }
                }
            }
            if (!group_sync(&group[2], gphase, abort, lim) || *abort) {
                ok = false;
                break;
            }
            if (wtid < N) {
                const int c = wtid;
                const double v = __ldcg(p.sums + static_cast<size_t>(I.unit) * N + c);
                const bool real = (c % W_PAD) < p.w && (c / W_PAD) < nheads;
                // log2 v = e + log2 f with v = f * 2^e, f in [1, 2) (v is a normal double: its
                // largest term is at least 2^-990)
                const unsigned long long bits = static_cast<unsigned long long>(__double_as_longlong(v));
                const int ex = static_cast<int>((bits >> 52) & 0x7FFull) - 1023;
                const float f = static_cast<float>(__longlong_as_double(static_cast<long long>(
                    (bits & 0x000FFFFFFFFFFFFFull) | 0x3FF0000000000000ull)));
                nlse_s[c] = real && v > 0.0 ? -(static_cast<float>(ex) + lg2_approx(f)) : -INFINITY;
            }
            if (!group_sync(&group[2], gphase, abort, lim)) {
                ok = false;
                break;
            }
            const float* nlse = nlse_s;
            // ---------------------------------------------------- the item's tiles
            for (int jt = 0; jt < n; ++jt, ++b_it) {
                const int acc = b_it % kAcc;
                if (!mbar_wait(&b_full[acc], (b_it / kAcc) & 1, abort, lim)) {
                    ok = false;
                    break;
                }
                tc_fence_after_sync();
                const int t = tile0 + jt;
                const int j = t * kTileKeys + eq * 32 + lane;
                const bool edge = (t * kTileKeys + kTileKeys - 1 >= P) || (t * kTileKeys + kTileKeys > L);
                const uint32_t taddr = tmem_base + lane_base + static_cast<uint32_t>((kAcc + acc) * N);
                float vv[N / 16][16];  // every 16-column chunk in flight, then one wait
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
#pragma unroll
                    for (int h = 0; h < kHeads; ++h)
                        if (h < nheads) out[h * T + j] = accum[h];
                }
            }
            // every warp is done with nlse_s before the next item's lse overwrites it
            if (!group_sync(&group[2], gphase, abort, lim)) {
                ok = false;
                break;
            }
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

template <int N, int W_PAD>
cudaError_t launch_one(const LayersParams& p, int grid, cudaStream_t stream) {
    auto kern = score_layers_kernel<N, W_PAD>;
    constexpr int smem = LayersSmem<N>::kDynamic;
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
    NvtxRange range("score_layers_kernel");
    return cudaLaunchKernelEx(&cfg, kern, p);
}

cudaError_t dispatch(const LayersParams& p, int n_cols, int w_pad, int grid, cudaStream_t st) {
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

cudaError_t launch_score_layers(const LayersLaunch& L, cudaStream_t stream) {
    static LayersParams p;  // ~30 KB, kept off the host stack; calls are serialised by `mu`
    static std::mutex mu;
    std::lock_guard<std::mutex> lock(mu);
    memset(&p, 0, sizeof(p));
    const int nl = static_cast<int>(L.layers.size());
    const int nb = static_cast<int>(L.batch_layer.size());
    const int ns = static_cast<int>(L.seq_start.size());
    const int nu = static_cast<int>(L.units.size()) - 1;  // the last entry closes the table
    if (nl < 1 || nl > kMaxLaunchLayers || nb < 1 || nb > kMaxLaunchBatches ||
        static_cast<int>(L.sel_heads.size()) > kMaxLaunchSel || ns < 1 || ns > kMaxLaunchSeqs ||
        nu < 0 || nu > kMaxLaunchUnits || L.grid < 1)
        return cudaErrorInvalidValue;
    if (nu == 0) return cudaSuccess;
    for (int l = 0; l < nl; ++l) {
        p.tmap_k[l] = L.layers[l].tmap_k;
        p.tmap_q[l] = L.layers[l].tmap_q;
        p.scores[l] = L.layers[l].scores;
        p.lse[l] = L.layers[l].lse;
        p.lse_stride[l] = L.layers[l].lse_stride;
    }
    p.cu_seqlens = L.cu_seqlens_dev;
    p.sums = L.sums;
    p.counters = L.counters;
    p.status = L.status;
    p.S = ns;
    p.T = L.T;
    p.w = L.w;
    p.n_units = nu;
    p.n_items = L.units[nu].item0;
    p.n_layers = nl;
    p.seq0 = L.seq0;
    p.S_all = L.S_all;
    p.cu_hash = L.cu_hash;
    p.sl2 = L.softmax_scale * 1.4426950408889634f;
    p.wait_cycles = wait_limit_cycles();
    for (int i = 0; i < nb; ++i) {
        p.batch_layer[i] = L.batch_layer[i];
        p.batch_group[i] = L.batch_group[i];
        p.batch_first[i] = L.batch_first[i];
        p.batch_nheads[i] = L.batch_nheads[i];
        p.batch_sel[i] = L.batch_sel[i];
    }
    for (size_t i = 0; i < L.sel_heads.size(); ++i) p.sel_heads[i] = L.sel_heads[i];
    for (int s = 0; s < ns; ++s) {
        p.seq_start[s] = L.seq_start[s];
        p.seq_len[s] = L.seq_len[s];
    }
    for (int u = 0; u <= nu; ++u) p.units[u] = L.units[u];
    if (p.n_items == 0) return cudaSuccess;
    const int grid = std::min(L.grid, p.n_items);
    if (L.given_lse) {  // one pass, no exchange: only the item counter
        const cudaError_t e = cudaMemsetAsync(L.counters + nu, 0, sizeof(int), stream);
        return e != cudaSuccess ? e : dispatch_lse_layers(p, L.n_cols, L.w_pad, grid, stream);
    }
    // the exchange's accumulators, its arrival counters and the item counter start at zero
    cudaError_t e = cudaMemsetAsync(L.sums, 0, static_cast<size_t>(nu) * L.n_cols * sizeof(double), stream);
    if (e == cudaSuccess) e = cudaMemsetAsync(L.counters, 0, static_cast<size_t>(nu + 1) * sizeof(int), stream);
    if (e != cudaSuccess) return e;
    return dispatch(p, L.n_cols, L.w_pad, grid, stream);
}

}  // namespace ckv
