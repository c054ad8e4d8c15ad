// Window-attention scoring (arxiv 2508.02401, Sec. 3.3 with the attention of Eq. 2):
//
//   a_h[j] = sum_{r < w, j <= P+r} exp(s_{h,r,j} - lse_{h,r}),   s_{h,r,j} = scale * q_{h,r}.k_j
//
// for every selected head h of a KV group, every window row r and every key j of a sequence
// (P = L - w).  The row normalisers lse need all keys before any probability can be summed
// over rows, so the work runs as two launches over the same decomposition:
//
//   pass 1: per chunk of keys, per window row: running (max, sum of 2^(x - max)) -> partials
//   pass 2: per chunk: combine the unit's partials into lse, recompute the logits and write
//           the window-summed probabilities a_h (the chunk's keys are usually still in L2).
//
// One CTA per SM, 256 threads, warp-specialised:
//   warp 0      TMA producer: streams 128-key x 128-dim bf16 tiles of K (two 128-byte-swizzled
//               64-column boxes) into a 6-stage shared-memory ring;
//   warp 1      allocates TMEM and issues tcgen05.mma (M = 128 keys, N = window rows of the
//               batch's heads, K = 128) into one of two TMEM accumulators;
//   warps 2-3   stage the unit's window query rows (the MMA's B operand) in shared memory;
//   warps 4-7   epilogue: each thread owns one key (one TMEM lane) and reads all of its
//               window-row logits, so both the per-row online softmax state (pass 1) and the
//               per-key sum over rows (pass 2) are thread-local.
//
// Work unit = (sequence, KV head, batch of up to 64/W_PAD selected heads); each unit's key
// tiles are split into chunks of `chunk_tiles` tiles (one chunk = one work item).
#include "ckv_device.cuh"
#include "ckv_internal.h"

namespace ckv {

struct alignas(128) ScoreParams {
    CUtensorMap tmap_k;            // K as {128 (dim), H_kv, T}, box {64, 1, 128}, 128B swizzle
    const __nv_bfloat16* q_win;    // [S, w, H_q, 128] packed
    const int32_t* cu_seqlens;     // device [S+1]
    float2* partials;              // [n_items, N]: (max, sum) per window-row column
    float* scores;                 // [n_sel, T]
    int* status;
    int S, T, Hq, w, nb, n_items, chunk_tiles, skip_le;
    uint32_t cu_hash;
    float sl2;                     // softmax scale * log2(e)
    int16_t batch_group[kMaxBatches];   // KV head of each head batch
    int16_t batch_first[kMaxBatches];   // score row of the batch's first head
    int16_t batch_nheads[kMaxBatches];  // heads in the batch
    int16_t sel_heads[kMaxQHeads];      // query head of each score row
};

struct Item {
    int s, seq_start, L, P, b, g, first, nheads, chunk, nchunks, tile0, tile1, unit_base;
};

constexpr int kStages = 6;
constexpr int kTileBytes = kTileKeys * kHeadDim * 2;  // 32 KiB
constexpr int kHalfBytes = kTileBytes / 2;            // 64 columns x 128 keys
constexpr float kLazyTau = 8.0f;                      // rescale only when 2^(x-m) > 2^8

// Maps a work item to its sequence, head batch and key-tile range by walking cu_seqlens.
// Returns false (and records an error) if the device lengths do not produce this item.
__device__ __forceinline__ bool decode_item(const ScoreParams& p, int item, Item& it) {
    int base = 0;
    for (int s = 0; s < p.S; ++s) {
        const int t0 = p.cu_seqlens[s], t1 = p.cu_seqlens[s + 1];
        const int L = t1 - t0;
        if (L < 0 || t0 < 0 || t1 > p.T) return false;
        const int tiles = (L + kTileKeys - 1) / kTileKeys;
        const int nch = (L > p.skip_le && L > 0) ? (tiles + p.chunk_tiles - 1) / p.chunk_tiles : 0;
        const int cnt = nch * p.nb;
        if (item < base + cnt) {
            const int rem = item - base;
            it.s = s;
            it.seq_start = t0;
            it.L = L;
            it.P = L - p.w;
            it.b = rem / nch;
            it.chunk = rem % nch;
            it.nchunks = nch;
            it.g = p.batch_group[it.b];
            it.first = p.batch_first[it.b];
            it.nheads = p.batch_nheads[it.b];
            it.tile0 = it.chunk * p.chunk_tiles;
            it.tile1 = min(tiles, it.tile0 + p.chunk_tiles);
            it.unit_base = item - it.chunk;
            return true;
        }
        base += cnt;
    }
    return false;
}

template <int N>
struct SmemLayout {
    static constexpr int kRing = 0;
    static constexpr int kQ = kRing + kStages * kTileBytes;
    static constexpr int kQHalf = N * 128;
    static constexpr int kBars = kQ + 2 * kQHalf;
    // full[kStages], empty[kStages], acc_full[2], acc_empty[2], q_full, q_empty, done
    static constexpr int kNumBars = 2 * kStages + 7;
    static constexpr int kRed = kBars + 8 * kNumBars;   // float2 [4][N]
    static constexpr int kLse = kRed + 8 * 4 * N;       // float [N]
    static constexpr int kTmemSlot = kLse + 4 * N;
    static constexpr int kAbort = kTmemSlot + 4;
    static constexpr int kBytes = kAbort + 4;
    static constexpr int kDynamic = kBytes + 1024;      // slack to align the base to 1024 B
};

template <int PASS, int N, int W_PAD>
__global__ void __launch_bounds__(256, 1) score_kernel(const __grid_constant__ ScoreParams p) {
    static_assert(N == 32 || N == 64, "N");
    static_assert(W_PAD == 8 || W_PAD == 16 || W_PAD == 32 || W_PAD == 64, "W_PAD");
    static_assert(W_PAD <= N, "a head's rows fit in one MMA");
    constexpr int HPB = N / W_PAD;  // heads per batch
    using SL = SmemLayout<N>;
    constexpr uint32_t kIdesc = idesc_bf16_f32(kTileKeys, N);

    extern __shared__ uint8_t smem_raw[];
    uint8_t* sm = reinterpret_cast<uint8_t*>(
        (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
    uint8_t* ring = sm + SL::kRing;
    uint8_t* qbuf = sm + SL::kQ;
    uint64_t* bars = reinterpret_cast<uint64_t*>(sm + SL::kBars);
    uint64_t* full = bars;
    uint64_t* empty = bars + kStages;
    uint64_t* acc_full = bars + 2 * kStages;
    uint64_t* acc_empty = acc_full + 2;
    uint64_t* q_full = acc_empty + 2;
    uint64_t* q_empty = q_full + 1;
    uint64_t* done = q_empty + 1;
    float2* red = reinterpret_cast<float2*>(sm + SL::kRed);
    float* lse_s = reinterpret_cast<float*>(sm + SL::kLse);
    uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(sm + SL::kTmemSlot);
    volatile int* abort = reinterpret_cast<volatile int*>(sm + SL::kAbort);

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;

    if (threadIdx.x == 0) {
        for (int i = 0; i < kStages; ++i) {
            mbar_init(&full[i], 1);
            mbar_init(&empty[i], 1);
        }
        for (int i = 0; i < 2; ++i) {
            mbar_init(&acc_full[i], 1);
            mbar_init(&acc_empty[i], 128);
        }
        mbar_init(q_full, 64);
        mbar_init(q_empty, 1);
        mbar_init(done, 1);
        *abort = 0;
        fence_mbar_init();
        tma_prefetch_desc(&p.tmap_k);
    }
    if (warp == 1) {
        tmem_alloc(tmem_slot, 2 * N);
        tmem_relinquish();
    }
    // Work items as the host counted them must match what the device lengths produce.
    if (blockIdx.x == 0 && threadIdx.x == 32 * 2) {
        int total = 0;
        bool ok = true;
        for (int s = 0; s < p.S; ++s) {
            const int L = p.cu_seqlens[s + 1] - p.cu_seqlens[s];
            if (L < 0 || p.cu_seqlens[s + 1] > p.T) ok = false;
            const int tiles = (L + kTileKeys - 1) / kTileKeys;
            total += (L > p.skip_le && L > 0) ? (tiles + p.chunk_tiles - 1) / p.chunk_tiles * p.nb : 0;
        }
        if (!ok || total != p.n_items || p.cu_seqlens[p.S] != p.T ||
            seqlens_hash(p.cu_seqlens, p.S) != p.cu_hash)
            record_error(p.status, kDevBadSeqlens, 100 + PASS);
    }
    tc_fence_before_sync();
    __syncthreads();
    tc_fence_after_sync();
    const uint32_t tmem_base = *tmem_slot;

    if (warp == 0) {
        // ------------------------------------------------------------ TMA producer
        if (lane == 0) {
            int it = 0;
            bool ok = true;
            for (int item = blockIdx.x; ok && item < p.n_items; item += gridDim.x) {
                Item I;
                if (!decode_item(p, item, I)) continue;
                for (int t = I.tile0; t < I.tile1; ++t, ++it) {
                    const int stage = it % kStages;
                    const uint32_t ph = (it / kStages) & 1;
                    if (!mbar_wait(&empty[stage], ph ^ 1, abort)) {
                        ok = false;
                        break;
                    }
                    mbar_arrive_expect_tx(&full[stage], kTileBytes);
                    uint8_t* dst = ring + stage * kTileBytes;
                    const int tok = I.seq_start + t * kTileKeys;
                    tma_load_3d(dst, &p.tmap_k, &full[stage], 0, I.g, tok);
                    tma_load_3d(dst + kHalfBytes, &p.tmap_k, &full[stage], 64, I.g, tok);
                }
            }
            if (!ok) {
                *abort = 1;
                record_error(p.status, kDevTimeout, 10 * PASS + 0);
            }
            // Let every issued copy land before the block may exit.
            const int n_issued = it;
            for (int k = n_issued - 1; k >= 0 && k >= n_issued - kStages; --k) {
                volatile int never = 0;
                mbar_wait(&full[k % kStages], (k / kStages) & 1, &never);
            }
        }
    } else if (warp == 1) {
        // ------------------------------------------------------------ MMA issuer
        if (lane == 0) {
            int it = 0, acc_it = 0, item_it = 0;
            bool ok = true;
            for (int item = blockIdx.x; ok && item < p.n_items; item += gridDim.x) {
                Item I;
                if (!decode_item(p, item, I)) continue;
                if (!mbar_wait(q_full, item_it & 1, abort)) {
                    ok = false;
                    break;
                }
                tc_fence_after_sync();
                for (int t = I.tile0; t < I.tile1; ++t, ++it, ++acc_it) {
                    const int stage = it % kStages;
                    const int acc = acc_it & 1;
                    if (!mbar_wait(&full[stage], (it / kStages) & 1, abort) ||
                        !mbar_wait(&acc_empty[acc], ((acc_it >> 1) & 1) ^ 1, abort)) {
                        ok = false;
                        break;
                    }
                    tc_fence_after_sync();
                    const uint32_t d_tmem = tmem_base + static_cast<uint32_t>(acc * N);
                    const uint32_t a0 = smem_u32(ring + stage * kTileBytes);
                    const uint32_t b0 = smem_u32(qbuf);
#pragma unroll
                    for (int kk = 0; kk < kHeadDim / 16; ++kk) {
                        const uint32_t koff = (kk & 3) * 32;
                        const uint64_t ad = sdesc_k_major_sw128(a0 + (kk >> 2) * kHalfBytes + koff);
                        const uint64_t bd = sdesc_k_major_sw128(b0 + (kk >> 2) * SL::kQHalf + koff);
                        umma_bf16(d_tmem, ad, bd, kIdesc, kk > 0 ? 1u : 0u);
                    }
                    umma_commit(&empty[stage]);
                    umma_commit(&acc_full[acc]);
                }
                if (!ok) break;
                umma_commit(q_empty);
                ++item_it;
            }
            if (!ok) {
                *abort = 1;
                record_error(p.status, kDevTimeout, 10 * PASS + 1);
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
        for (int item = blockIdx.x; item < p.n_items; item += gridDim.x) {
            Item I;
            if (!decode_item(p, item, I)) continue;
            if (!mbar_wait(q_empty, (item_it & 1) ^ 1, abort)) {
                *abort = 1;
                record_error(p.status, kDevTimeout, 10 * PASS + 2);
                break;
            }
            // Each thread owns one 16-byte column chunk c of rows r0, r0+4, ...: all of its
            // loads are issued before any store, so their latencies overlap.
            constexpr int kPer = N * 16 / 64;
            const int c = tid & 15, r0 = tid >> 4;
            uint4 vals[kPer];
#pragma unroll
            for (int i = 0; i < kPer; ++i) {
                const int r = r0 + 4 * i;
                const int slot = r / W_PAD, rr = r % W_PAD;
                vals[i] = make_uint4(0u, 0u, 0u, 0u);
                if (slot < I.nheads && rr < p.w) {
                    const int h = p.sel_heads[I.first + slot];
                    const uint4* src = reinterpret_cast<const uint4*>(
                        p.q_win + ((static_cast<size_t>(I.s) * p.w + rr) * p.Hq + h) * kHeadDim);
                    vals[i] = __ldg(src + c);
                }
            }
#pragma unroll
            for (int i = 0; i < kPer; ++i) {
                const int r = r0 + 4 * i;
                const int half = c >> 3, cc = c & 7;
                *reinterpret_cast<uint4*>(qbuf + half * SL::kQHalf + r * 128 +
                                          ((cc ^ (r & 7)) << 4)) = vals[i];
            }
            fence_proxy_async_smem();
            mbar_arrive(q_full);
            ++item_it;
        }
    } else {
        // ------------------------------------------------------------ epilogue
        const int eq = warp - 4;           // TMEM lane quarter
        const int tid = threadIdx.x - 128;
        int acc_it = 0;
        bool ok = true;
        for (int item = blockIdx.x; ok && item < p.n_items; item += gridDim.x) {
            Item I;
            if (!decode_item(p, item, I)) continue;
            uint64_t colmask = 0;
#pragma unroll
            for (int c = 0; c < N; ++c)
                if ((c % W_PAD) < p.w && (c / W_PAD) < I.nheads) colmask |= 1ull << c;
            const bool all_cols = colmask == (N == 64 ? ~0ull : ((1ull << N) - 1));

            float st_a[N];  // pass 1: running max (log2 units); pass 2: lse (log2 units)
            float st_b[N];  // pass 1: running sum relative to st_a
            if constexpr (PASS == 1) {
#pragma unroll
                for (int c = 0; c < N; ++c) {  // set from the first tile below
                    st_a[c] = -1e30f;
                    st_b[c] = 0.f;
                }
            } else {
                named_bar_sync(1, 128);  // previous item's readers of lse_s are done
                if (tid < N) {
                    float M = -INFINITY, S = 0.f;
                    const int n = min(I.nchunks, p.n_items - I.unit_base);
                    const float2* src = p.partials + static_cast<size_t>(I.unit_base) * N + tid;
                    int k = 0;
                    for (; k + 4 <= n; k += 4) {  // four independent loads in flight
                        float2 pr[4];
#pragma unroll
                        for (int u = 0; u < 4; ++u) pr[u] = src[static_cast<size_t>(k + u) * N];
#pragma unroll
                        for (int u = 0; u < 4; ++u) {
                            const float Mn = fmaxf(M, pr[u].x);
                            S = S * ex2_approx(M - Mn) + pr[u].y * ex2_approx(pr[u].x - Mn);
                            M = Mn;
                        }
                    }
                    for (; k < n; ++k) {
                        const float2 pr = src[static_cast<size_t>(k) * N];
                        const float Mn = fmaxf(M, pr.x);
                        S = S * ex2_approx(M - Mn) + pr.y * ex2_approx(pr.x - Mn);
                        M = Mn;
                    }
                    lse_s[tid] = M + log2f(S);
                }
                named_bar_sync(1, 128);
#pragma unroll
                for (int c = 0; c < N; ++c) st_a[c] = lse_s[c];
            }

            for (int t = I.tile0; t < I.tile1; ++t, ++acc_it) {
                const int acc = acc_it & 1;
                if (!mbar_wait(&acc_full[acc], (acc_it >> 1) & 1, abort)) {
                    ok = false;
                    break;
                }
                tc_fence_after_sync();
                const uint32_t taddr = tmem_base + (static_cast<uint32_t>(eq * 32) << 16) +
                                       static_cast<uint32_t>(acc * N);
                const int j = t * kTileKeys + eq * 32 + lane;  // sequence-local key position
                const bool edge = (t * kTileKeys + kTileKeys - 1 >= I.P) ||
                                  (t * kTileKeys + kTileKeys > I.L);
                const bool simple = all_cols && !edge;
                const bool key_ok = j < I.L;
                const int jr = j - I.P;  // row r sees key j iff r >= jr
                const bool first = t == I.tile0;
                float accum[HPB];
#pragma unroll
                for (int h = 0; h < HPB; ++h) accum[h] = 0.f;

#pragma unroll
                for (int cc = 0; cc < N / 32; ++cc) {
                    float v[32];
                    tmem_ld32(taddr + cc * 32, v);
                    if (cc == N / 32 - 1) {  // the accumulator is free for the next tile
                        tc_fence_before_sync();
                        mbar_arrive(&acc_empty[acc]);
                    }
                    if constexpr (PASS == 1) {
                        if (first) {
                            // The thread's first key of the item seeds each row's running
                            // maximum.  A row that cannot see this key cannot see the thread's
                            // later keys either (they lie further right), so it stays empty.
#pragma unroll
                            for (int i = 0; i < 32; ++i) {
                                const int c = cc * 32 + i;
                                const bool valid = simple || (((colmask >> c) & 1ull) && key_ok &&
                                                              (c % W_PAD) >= jr);
                                st_a[c] = valid ? v[i] * p.sl2 : -1e30f;
                                st_b[c] = valid ? 1.f : 0.f;
                            }
                            continue;
                        }
                        float dmax = -INFINITY;
#pragma unroll
                        for (int i = 0; i < 32; ++i) {
                            const int c = cc * 32 + i;
                            float d = fmaf(v[i], p.sl2, -st_a[c]);
                            if (!simple) {
                                const bool valid = ((colmask >> c) & 1ull) && key_ok && (c % W_PAD) >= jr;
                                d = valid ? d : -INFINITY;
                            }
                            v[i] = d;
                            dmax = fmaxf(dmax, d);
                        }
                        if (dmax > kLazyTau) {  // a new running maximum well above the old one
#pragma unroll
                            for (int i = 0; i < 32; ++i) {
                                const int c = cc * 32 + i;
                                if (v[i] > kLazyTau) {
                                    st_b[c] *= ex2_approx(-v[i]);
                                    st_a[c] += v[i];
                                    v[i] = 0.f;
                                }
                            }
                        }
#pragma unroll
                        for (int i = 0; i < 32; ++i) st_b[cc * 32 + i] += ex2_approx(v[i]);
                    } else {
#pragma unroll
                        for (int i = 0; i < 32; ++i) {
                            const int c = cc * 32 + i;
                            float e = ex2_approx(fmaf(v[i], p.sl2, -st_a[c]));
                            if (!simple) {
                                const bool valid = ((colmask >> c) & 1ull) && key_ok && (c % W_PAD) >= jr;
                                e = valid ? e : 0.f;
                            }
                            accum[c / W_PAD] += e;
                        }
                    }
                }
                if constexpr (PASS == 2) {
                    if (key_ok) {
                        const size_t col = static_cast<size_t>(I.seq_start) + j;
#pragma unroll
                        for (int h = 0; h < HPB; ++h)
                            if (h < I.nheads)
                                p.scores[static_cast<size_t>(I.first + h) * p.T + col] = accum[h];
                    }
                }
            }
            if (!ok) break;

            if constexpr (PASS == 1) {
                // Combine the 128 threads' (max, sum) per column and write the chunk partial.
                // Level-major butterflies over 32 columns at a time, so the shuffles of
                // different columns overlap instead of forming one long dependent chain.
#pragma unroll
                for (int hc = 0; hc < N / 32; ++hc) {
                    float M[32];
#pragma unroll
                    for (int i = 0; i < 32; ++i) M[i] = st_a[hc * 32 + i];
#pragma unroll
                    for (int o = 16; o > 0; o >>= 1)
#pragma unroll
                        for (int i = 0; i < 32; ++i)
                            M[i] = fmaxf(M[i], __shfl_xor_sync(0xffffffffu, M[i], o));
#pragma unroll
                    for (int i = 0; i < 32; ++i) st_b[hc * 32 + i] *= ex2_approx(st_a[hc * 32 + i] - M[i]);
#pragma unroll
                    for (int o = 16; o > 0; o >>= 1)
#pragma unroll
                        for (int i = 0; i < 32; ++i)
                            st_b[hc * 32 + i] += __shfl_xor_sync(0xffffffffu, st_b[hc * 32 + i], o);
                    if (lane == 0) {
#pragma unroll
                        for (int i = 0; i < 32; ++i)
                            red[eq * N + hc * 32 + i] = make_float2(M[i], st_b[hc * 32 + i]);
                    }
                }
                named_bar_sync(1, 128);
                if (tid < N) {
                    float M = red[tid].x;
#pragma unroll
                    for (int q = 1; q < 4; ++q) M = fmaxf(M, red[q * N + tid].x);
                    float S = 0.f;
#pragma unroll
                    for (int q = 0; q < 4; ++q) S += red[q * N + tid].y * ex2_approx(red[q * N + tid].x - M);
                    p.partials[static_cast<size_t>(item) * N + tid] = make_float2(M, S);
                }
                named_bar_sync(1, 128);
            }
        }
        if (!ok) {
            *abort = 1;
            record_error(p.status, kDevTimeout, 10 * PASS + 3);
        }
    }

    tc_fence_before_sync();
    __syncthreads();
    if (warp == 1) {
        tc_fence_after_sync();
        tmem_dealloc(tmem_base, 2 * N);
    }
}

// ------------------------------------------------------------------------------ host side
namespace {

template <int PASS, int N, int W_PAD>
cudaError_t launch_one(const ScoreParams& p, int grid, cudaStream_t stream) {
    auto kern = score_kernel<PASS, N, W_PAD>;
    constexpr int smem = SmemLayout<N>::kDynamic;
    static bool configured = false;  // benign race: the attribute call is idempotent
    if (!configured) {
        cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
        if (e != cudaSuccess) return e;
        configured = true;
    }
    kern<<<grid, 256, smem, stream>>>(p);
    return cudaGetLastError();
}

template <int PASS>
cudaError_t dispatch(const ScoreParams& p, int n_cols, int w_pad, int grid, cudaStream_t st) {
    if (n_cols == 32) {
        if (w_pad == 8) return launch_one<PASS, 32, 8>(p, grid, st);
        if (w_pad == 16) return launch_one<PASS, 32, 16>(p, grid, st);
        if (w_pad == 32) return launch_one<PASS, 32, 32>(p, grid, st);
    } else if (n_cols == 64) {
        if (w_pad == 8) return launch_one<PASS, 64, 8>(p, grid, st);
        if (w_pad == 16) return launch_one<PASS, 64, 16>(p, grid, st);
        if (w_pad == 32) return launch_one<PASS, 64, 32>(p, grid, st);
        if (w_pad == 64) return launch_one<PASS, 64, 64>(p, grid, st);
    }
    return cudaErrorInvalidValue;
}

}  // namespace

cudaError_t launch_score(const ScoreLaunch& L, cudaStream_t stream) {
    static_assert(sizeof(ScoreParams) < 4096, "kernel parameters");
    ScoreParams p;
    memset(&p, 0, sizeof(p));
    p.tmap_k = L.tmap_k;
    p.q_win = reinterpret_cast<const __nv_bfloat16*>(L.q_win);
    p.cu_seqlens = L.cu_seqlens_dev;
    p.partials = reinterpret_cast<float2*>(L.partials);
    p.scores = L.scores;
    p.status = L.status;
    p.S = L.S;
    p.T = L.T;
    p.Hq = L.Hq;
    p.w = L.w;
    p.nb = L.nb;
    p.n_items = L.n_items;
    p.chunk_tiles = L.chunk_tiles;
    p.skip_le = L.skip_le;
    p.cu_hash = L.cu_hash;
    p.sl2 = L.softmax_scale * 1.4426950408889634f;
    for (int b = 0; b < L.nb; ++b) {
        p.batch_group[b] = static_cast<int16_t>(L.batch_group[b]);
        p.batch_first[b] = static_cast<int16_t>(L.batch_first[b]);
        p.batch_nheads[b] = static_cast<int16_t>(L.batch_nheads[b]);
    }
    for (int i = 0; i < L.n_sel; ++i) p.sel_heads[i] = static_cast<int16_t>(L.sel_heads[i]);
    if (L.n_items == 0) return cudaSuccess;
    const int grid = L.n_items < L.grid ? L.n_items : L.grid;
    cudaError_t e = dispatch<1>(p, L.n_cols, L.w_pad, grid, stream);
    if (e != cudaSuccess || !L.scores) return e;
    return dispatch<2>(p, L.n_cols, L.w_pad, grid, stream);
}

int score_partials_stride(int n_cols) { return n_cols; }

}  // namespace ckv
