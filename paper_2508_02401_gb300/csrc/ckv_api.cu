// The C ABI declared in include/ckv.h: argument validation (all on the host, before anything
// is enqueued), per-layer planning of the head batches and key chunks, the workspace layout,
// TMA descriptor set-up and kernel dispatch.
#include <math.h>
#include <stdarg.h>
#include <stdio.h>
#include <string.h>

#include <algorithm>
#include <mutex>
#include <vector>

#include "ckv.h"
#include "ckv_device.cuh"
#include "ckv_internal.h"

#include <limits.h>

#include <atomic>

namespace ckv {
namespace {

thread_local char g_msg[512] = "";

ckv_status fail(ckv_status st, const char* fmt, ...) {
    va_list ap;
    va_start(ap, fmt);
    vsnprintf(g_msg, sizeof g_msg, fmt, ap);
    va_end(ap);
    return st;
}

ckv_status cuda_fail(cudaError_t e, const char* what) {
    return fail(CKV_ERR_CUDA, "%s: %s (%s)", what, cudaGetErrorName(e), cudaGetErrorString(e));
}

bool aligned(const void* p, size_t a) { return (reinterpret_cast<uintptr_t>(p) % a) == 0; }

constexpr size_t kWsAlign = 256;

size_t round_up(size_t x, size_t a) { return (x + a - 1) / a * a; }

// Everything a call needs to know about one layer of the config.
struct Plan {
    int Hq = 0, Hkv = 0, G = 0, w = 0, w_pad = 0, n_cols = 0, hpb = 0, budget = 0, max_ctas = 0;
    int score_path = CKV_SCORE_AUTO;
    int n_sel = 0, nb = 0;
    int scope = CKV_SCOPE_KV_HEAD, n_vec = 0;  // selections per sequence: H_kv or 1
    // group_first: first score row of each selection's heads (n_vec + 1 entries)
    float scale = 0.f;
    std::vector<int> sel_heads, batch_group, batch_first, batch_nheads, group_first;
};

ckv_status check_config(const ckv_config* cfg) {
    if (!cfg) return fail(CKV_ERR_INVALID_ARG, "cfg is NULL");
    if (cfg->num_layers < 1) return fail(CKV_ERR_INVALID_ARG, "num_layers %d < 1", cfg->num_layers);
    if (cfg->num_kv_heads < 1 || cfg->num_q_heads < 1)
        return fail(CKV_ERR_INVALID_ARG, "head counts must be positive");
    if (cfg->num_q_heads % cfg->num_kv_heads != 0)
        return fail(CKV_ERR_INVALID_ARG, "num_q_heads %d is not a multiple of num_kv_heads %d",
                    cfg->num_q_heads, cfg->num_kv_heads);
    if (cfg->num_q_heads > kMaxQHeads)
        return fail(CKV_ERR_UNSUPPORTED, "num_q_heads %d > %d", cfg->num_q_heads, kMaxQHeads);
    if (cfg->head_dim <= 0) return fail(CKV_ERR_INVALID_ARG, "head_dim %d", cfg->head_dim);
    if (cfg->head_dim != kHeadDim)
        return fail(CKV_ERR_UNSUPPORTED, "head_dim %d (only 128 is supported)", cfg->head_dim);
    if (cfg->window < 1) return fail(CKV_ERR_INVALID_ARG, "window %d < 1", cfg->window);
    if (cfg->window > kMaxWindow)
        return fail(CKV_ERR_UNSUPPORTED, "window %d > %d", cfg->window, kMaxWindow);
    if (cfg->pool_kernel < 1 || cfg->pool_kernel % 2 == 0)
        return fail(CKV_ERR_INVALID_ARG, "pool_kernel %d must be odd and >= 1", cfg->pool_kernel);
    if (cfg->pool_kernel > kMaxPoolKernel)
        return fail(CKV_ERR_UNSUPPORTED, "pool_kernel %d > %d", cfg->pool_kernel, kMaxPoolKernel);
    if (cfg->pool_type != CKV_POOL_MAX && cfg->pool_type != CKV_POOL_AVG)
        return fail(CKV_ERR_INVALID_ARG, "pool_type %d", cfg->pool_type);
    if (cfg->head_order != CKV_POOL_THEN_SUM && cfg->head_order != CKV_SUM_THEN_POOL)
        return fail(CKV_ERR_INVALID_ARG, "head_order %d", cfg->head_order);
    if (!(cfg->softmax_scale >= 0.f) || !isfinite(cfg->softmax_scale))
        return fail(CKV_ERR_INVALID_ARG, "softmax_scale must be finite and >= 0");
    if (cfg->max_ctas < 0) return fail(CKV_ERR_INVALID_ARG, "max_ctas %d < 0", cfg->max_ctas);
    if (cfg->score_path < CKV_SCORE_AUTO || cfg->score_path > CKV_SCORE_RELOAD)
        return fail(CKV_ERR_INVALID_ARG, "score_path %d", cfg->score_path);
    if (cfg->scope != CKV_SCOPE_KV_HEAD && cfg->scope != CKV_SCOPE_LAYER)
        return fail(CKV_ERR_INVALID_ARG, "scope %d", cfg->scope);
    if (!cfg->head_mask || !cfg->budgets)
        return fail(CKV_ERR_INVALID_ARG, "head_mask and budgets must be host pointers");
    return CKV_OK;
}

ckv_status make_plan(const ckv_config* cfg, int32_t layer, Plan& pl) {
    ckv_status st = check_config(cfg);
    if (st) return st;
    if (layer < 0 || layer >= cfg->num_layers)
        return fail(CKV_ERR_INVALID_ARG, "layer %d outside [0, %d)", layer, cfg->num_layers);
    pl.Hq = cfg->num_q_heads;
    pl.Hkv = cfg->num_kv_heads;
    pl.G = pl.Hq / pl.Hkv;
    pl.w = cfg->window;
    pl.budget = cfg->budgets[layer];
    pl.max_ctas = cfg->max_ctas;
    pl.score_path = cfg->score_path;
    if (pl.budget < pl.w)
        return fail(CKV_ERR_INVALID_ARG, "budget %d of layer %d is below the window %d", pl.budget,
                    layer, pl.w);
    pl.scale = cfg->softmax_scale > 0.f ? cfg->softmax_scale : 1.0f / sqrtf(static_cast<float>(kHeadDim));
    pl.w_pad = 8;
    while (pl.w_pad < pl.w) pl.w_pad *= 2;
    pl.hpb = kMaxCols / pl.w_pad;
    const uint8_t* mask = cfg->head_mask + static_cast<size_t>(layer) * pl.Hq;
    pl.scope = cfg->scope;
    pl.n_vec = pl.scope == CKV_SCOPE_LAYER ? 1 : pl.Hkv;
    pl.group_first.assign(pl.n_vec + 1, 0);
    int max_heads = 0;
    for (int g = 0; g < pl.Hkv; ++g) {
        if (pl.scope == CKV_SCOPE_KV_HEAD) pl.group_first[g] = pl.n_sel;
        std::vector<int> heads;
        for (int h = g * pl.G; h < (g + 1) * pl.G; ++h)
            if (mask[h]) heads.push_back(h);
        if (heads.empty() && pl.scope == CKV_SCOPE_KV_HEAD)
            return fail(CKV_ERR_INVALID_ARG, "KV group %d of layer %d has no selected head", g, layer);
        for (size_t i = 0; i < heads.size(); i += pl.hpb) {
            const int n = std::min<int>(pl.hpb, static_cast<int>(heads.size() - i));
            pl.batch_group.push_back(g);
            pl.batch_first.push_back(pl.n_sel + static_cast<int>(i));
            pl.batch_nheads.push_back(n);
            max_heads = std::max(max_heads, n);
        }
        for (int h : heads) pl.sel_heads.push_back(h);
        pl.n_sel += static_cast<int>(heads.size());
    }
    if (pl.n_sel == 0) return fail(CKV_ERR_INVALID_ARG, "layer %d has no selected head", layer);
    pl.group_first[pl.n_vec] = pl.n_sel;  // per layer: rows [0, n_sel) form one selection
    pl.nb = static_cast<int>(pl.batch_group.size());
    if (pl.nb > kMaxBatches) return fail(CKV_ERR_UNSUPPORTED, "too many head batches (%d)", pl.nb);
    pl.n_cols = (max_heads * pl.w_pad <= 32) ? 32 : 64;
    return CKV_OK;
}

ckv_status check_batch(const ckv_batch* b, int* T_out) {
    if (!b) return fail(CKV_ERR_INVALID_ARG, "batch is NULL");
    if (b->num_seqs < 1) return fail(CKV_ERR_INVALID_ARG, "num_seqs %d < 1", b->num_seqs);
    if (!b->cu_seqlens_host || !b->cu_seqlens_dev)
        return fail(CKV_ERR_INVALID_ARG, "cu_seqlens_host and cu_seqlens_dev are required");
    if (b->cu_seqlens_host[0] != 0) return fail(CKV_ERR_INVALID_ARG, "cu_seqlens[0] != 0");
    for (int s = 0; s < b->num_seqs; ++s)
        if (b->cu_seqlens_host[s + 1] < b->cu_seqlens_host[s])
            return fail(CKV_ERR_INVALID_ARG, "cu_seqlens decreases at %d", s);
    *T_out = b->cu_seqlens_host[b->num_seqs];
    return CKV_OK;
}

int64_t keep_total(const ckv_batch* b, int budget) {
    int64_t t = 0;
    for (int s = 0; s < b->num_seqs; ++s)
        t += std::min(budget, b->cu_seqlens_host[s + 1] - b->cu_seqlens_host[s]);
    return t;
}

// Work of the TMEM-resident scoring kernel (score_resident.cu): splits every (sequence, head
// batch) unit's key tiles into items of at most `c` tiles (c <= 512 / n_cols, so that an
// item's logits fit in TMEM) and packs units whole into rounds of at most `ctas` items; `c`
// minimises an estimate of the launch's time in tile loads per CTA.  While an item waits for
// its unit's exchange and runs pass 2, the next item's MMAs can fill the accumulators it
// leaves free and the ring can hold `ring` more tiles; a round costs its item length plus
// whatever of the exchange those do not cover.  CKV_ERR_UNSUPPORTED if a unit does not fit
// one round.
ckv_status plan_score(const Plan& pl, const ckv_batch* b, int skip_le, int ctas, ScoreLaunch& L,
                      int max_items_per_launch) {
    struct RawUnit {
        int seq, start, len, batch, tiles;
    };
    std::vector<RawUnit> raw;
    int max_tiles = 0;
    for (int s = 0; s < b->num_seqs; ++s) {
        const int t0 = b->cu_seqlens_host[s];
        const int len = b->cu_seqlens_host[s + 1] - t0;
        if (len <= skip_le || len <= 0) continue;
        const int tiles = (len + kTileKeys - 1) / kTileKeys;
        max_tiles = std::max(max_tiles, tiles);
        for (int bt = 0; bt < pl.nb; ++bt) raw.push_back({s, t0, len, bt, tiles});
    }
    L.items.clear();
    L.units.clear();
    L.slices.clear();
    L.resident = true;
    if (raw.empty()) return CKV_OK;
    if (b->num_seqs > 65535) return fail(CKV_ERR_UNSUPPORTED, "more than 65535 sequences");
    const int c_res = 512 / pl.n_cols;
    if (static_cast<long long>(max_tiles) > static_cast<long long>(c_res) * ctas)
        return fail(CKV_ERR_UNSUPPORTED,
                    "resident scoring: a sequence of %d key tiles needs items of at most %d tiles "
                    "on at least %d CTAs (%d available)", max_tiles, c_res,
                    (max_tiles + c_res - 1) / c_res, ctas);
    constexpr double kResExchange = 8.0;  // publish, exchange, combine and pass 2 from TMEM
    const int ring = pl.n_cols == 64 ? 5 : 6;
    const int c_hi = std::min(max_tiles, c_res);
    int best_c = -1;
    double best_cost = 0;
    for (int c = 1; c <= c_hi; ++c) {
        long long rounds = 0;
        int cur = 0;
        bool feasible = c <= 65535;
        for (const RawUnit& u : raw) {
            const int n = (u.tiles + c - 1) / c;
            if (n > ctas) {
                feasible = false;
                break;
            }
            if (cur + n > ctas) {
                ++rounds;
                cur = 0;
            }
            cur += n;
        }
        if (!feasible) continue;
        rounds += cur > 0;
        const double per_round = c + std::max(0.0, kResExchange - (c_res - c) - ring);
        const double cost = rounds * per_round + kResExchange;
        if (best_c < 0 || cost < best_cost) {
            best_c = c;
            best_cost = cost;
        }
    }
    if (best_c < 0) return fail(CKV_ERR_UNSUPPORTED, "cannot partition the scoring work");
    // Rounds of units; the grid is the largest round.
    std::vector<std::vector<int>> rounds(1);
    std::vector<int> round_items(1, 0);
    for (int ui = 0; ui < static_cast<int>(raw.size()); ++ui) {
        const int n = (raw[ui].tiles + best_c - 1) / best_c;
        if (round_items.back() + n > ctas) {
            rounds.emplace_back();
            round_items.push_back(0);
        }
        rounds.back().push_back(ui);
        round_items.back() += n;
    }
    const int grid = *std::max_element(round_items.begin(), round_items.end());
    if (grid > max_items_per_launch) return fail(CKV_ERR_UNSUPPORTED, "scoring grid too large");
    L.grid = grid;
    // Slices of consecutive rounds that fit one launch's item and unit tables.
    ScoreSlice cur{0, 0, 0, 0};
    for (size_t r = 0; r < rounds.size(); ++r) {
        const int nu = static_cast<int>(rounds[r].size());
        if (cur.n_rounds > 0 && ((cur.n_rounds + 1) * grid > max_items_per_launch ||
                                 cur.n_units + nu > kMaxScoreUnits)) {
            L.slices.push_back(cur);
            cur = ScoreSlice{static_cast<int>(L.items.size()), 0, static_cast<int>(L.units.size()), 0};
        }
        if (nu > kMaxScoreUnits) return fail(CKV_ERR_UNSUPPORTED, "too many scoring units in a round");
        int slot = 0;
        for (int ui : rounds[r]) {
            const RawUnit& u = raw[ui];
            const int n = (u.tiles + best_c - 1) / best_c;
            ScoreUnit su;
            su.seq_start = u.start;
            su.len = u.len;
            su.seq = static_cast<uint16_t>(u.seq);
            su.batch = static_cast<uint16_t>(u.batch);
            su.first_item = static_cast<uint16_t>(cur.n_rounds * grid + slot);
            su.nitems = static_cast<uint16_t>(n);
            const int uidx = cur.n_units;
            L.units.push_back(su);
            ++cur.n_units;
            for (int k = 0; k < n; ++k, ++slot) {
                ScoreItem it;
                it.unit = static_cast<uint16_t>(uidx);
                it.tile0 = static_cast<uint32_t>(k * best_c);
                it.ntiles = static_cast<uint16_t>(std::min(best_c, u.tiles - k * best_c));
                L.items.push_back(it);
            }
        }
        for (; slot < grid; ++slot) L.items.push_back(ScoreItem{0, 0, 0});
        ++cur.n_rounds;
    }
    L.slices.push_back(cur);
    return CKV_OK;
}

// Work of the single-pass kernel (window-row lse given): no exchange between CTAs, so the key
// tiles of all (sequence, head batch) units, taken in order, are cut into `grid` runs of
// (nearly) equal length, one per CTA; a run that crosses units becomes one item per unit.
// Round r of the item table holds every CTA's r-th item.
ckv_status plan_score_stream(const Plan& pl, const ckv_batch* b, int skip_le, int ctas, ScoreLaunch& L,
                             int max_items_per_launch) {
    struct RawUnit {
        int seq, start, len, batch, tiles;
    };
    std::vector<RawUnit> raw;
    int64_t total = 0;
    for (int s = 0; s < b->num_seqs; ++s) {
        const int t0 = b->cu_seqlens_host[s];
        const int len = b->cu_seqlens_host[s + 1] - t0;
        if (len <= skip_le || len <= 0) continue;
        const int tiles = (len + kTileKeys - 1) / kTileKeys;
        for (int bt = 0; bt < pl.nb; ++bt) {
            raw.push_back({s, t0, len, bt, tiles});
            total += tiles;
        }
    }
    L.items.clear();
    L.units.clear();
    L.slices.clear();
    L.resident = false;
    if (raw.empty()) return CKV_OK;
    if (b->num_seqs > 65535) return fail(CKV_ERR_UNSUPPORTED, "more than 65535 sequences");
    const int grid = static_cast<int>(std::min<int64_t>(ctas, total));
    const int64_t per = (total + grid - 1) / grid;
    if (per > 65535) return fail(CKV_ERR_UNSUPPORTED, "more than 65535 key tiles per CTA");
    struct Run {
        int raw;         // index into raw
        ScoreItem item;  // unit filled in per slice
    };
    std::vector<std::vector<Run>> runs(grid);
    int cta = 0;
    int64_t filled = 0;
    for (int ui = 0; ui < static_cast<int>(raw.size()); ++ui) {
        for (int t = 0; t < raw[ui].tiles;) {
            const int take = static_cast<int>(std::min<int64_t>(raw[ui].tiles - t, per - filled));
            runs[cta].push_back({ui, ScoreItem{0, static_cast<uint16_t>(take), static_cast<uint32_t>(t)}});
            t += take;
            filled += take;
            if (filled == per && cta + 1 < grid) {
                ++cta;
                filled = 0;
            }
        }
    }
    size_t rounds = 0;
    for (const auto& r : runs) rounds = std::max(rounds, r.size());
    L.grid = grid;
    const int max_rounds = std::max(1, max_items_per_launch / grid);
    std::vector<int> local(raw.size(), -1);
    size_t r = 0;
    while (r < rounds) {
        ScoreSlice sl{static_cast<int>(L.items.size()), 0, static_cast<int>(L.units.size()), 0};
        std::vector<int> used;
        while (r < rounds && sl.n_rounds < max_rounds) {
            int fresh = 0;
            for (int c = 0; c < grid; ++c)
                if (r < runs[c].size() && local[runs[c][r].raw] < 0) ++fresh;  // an upper bound
            if (sl.n_rounds > 0 && sl.n_units + fresh > kMaxScoreUnits) break;
            for (int c = 0; c < grid; ++c) {
                ScoreItem it{0, 0, 0};
                if (r < runs[c].size()) {
                    const int ui = runs[c][r].raw;
                    if (local[ui] < 0) {
                        if (sl.n_units >= kMaxScoreUnits)
                            return fail(CKV_ERR_UNSUPPORTED, "too many scoring units in a round");
                        local[ui] = sl.n_units++;
                        used.push_back(ui);
                        ScoreUnit su;
                        su.seq_start = raw[ui].start;
                        su.len = raw[ui].len;
                        su.seq = static_cast<uint16_t>(raw[ui].seq);
                        su.batch = static_cast<uint16_t>(raw[ui].batch);
                        su.first_item = 0;  // no exchange: unused
                        su.nitems = 0;
                        L.units.push_back(su);
                    }
                    it = runs[c][r].item;
                    it.unit = static_cast<uint16_t>(local[ui]);
                }
                L.items.push_back(it);
            }
            ++sl.n_rounds;
            ++r;
        }
        for (int ui : used) local[ui] = -1;
        L.slices.push_back(sl);
    }
    return CKV_OK;
}

struct WsLayout {
    size_t header = 0, partials = 0, counters = 0, sums = 0, unit_counters = 0, scores = 0,
           pooled = 0, srs_lse = 0;
    size_t hist = 0, arrivals = 0, chunk_start = 0, buckets = 0, info = 0, chunk_off = 0, total = 0;
    int max_chunks = 0;
};

int max_seqlen(const ckv_batch* b) {
    int m = 0;
    for (int s = 0; s < b->num_seqs; ++s)
        m = std::max(m, b->cu_seqlens_host[s + 1] - b->cu_seqlens_host[s]);
    return m;
}

WsLayout ws_layout(const Plan& pl, const ckv_batch* b, int T) {
    WsLayout l;
    const size_t units = static_cast<size_t>(b->num_seqs) * pl.n_vec;
    l.max_chunks = select_chunks(max_seqlen(b));
    size_t off = round_up(sizeof(WsHeader), kWsAlign);
    l.partials = off;
    off = round_up(off + static_cast<size_t>(kMaxScoreItems) * kMaxCols * sizeof(float2), kWsAlign);
    l.counters = off;
    off = round_up(off + kMaxScoreUnits * sizeof(int), kWsAlign);
    // the two-pass kernel's exchange: per (head batch, sequence) unit, an fp64 sum per column
    // and an arrival counter
    const size_t score_units = static_cast<size_t>(pl.nb) * b->num_seqs;
    l.sums = off;
    off = round_up(off + score_units * kMaxCols * sizeof(double), kWsAlign);
    l.unit_counters = off;  // and, after them, the kernel's item counter
    off = round_up(off + (score_units + 1) * sizeof(int), kWsAlign);
    l.scores = off;
    off = round_up(off + static_cast<size_t>(pl.n_sel) * T * sizeof(float), kWsAlign);
    l.pooled = off;
    off = round_up(off + static_cast<size_t>(pl.n_vec) * T * sizeof(float), kWsAlign);
    l.hist = off;  // zero outside a call: the selection leaves it as it found it
    off = round_up(off + units * select_hist_ints() * sizeof(int), kWsAlign);
    l.arrivals = off;  // zero outside a call, like hist
    off = round_up(off + units * sizeof(int), kWsAlign);
    l.chunk_start = off;
    off = round_up(off + units * l.max_chunks * select_hist_ints() * sizeof(int), kWsAlign);
    l.buckets = off;
    off = round_up(off + units * l.max_chunks * select_chunk_positions() * 8, kWsAlign);
    l.info = off;
    off = round_up(off + units * 4 * sizeof(int), kWsAlign);
    l.chunk_off = off;
    off = round_up(off + units * l.max_chunks * sizeof(int), kWsAlign);
    l.srs_lse = off;  // ckv_semantic_retrieval_scores: the masked lse of the decode rows
    off = round_up(off + static_cast<size_t>(pl.Hq) * b->num_seqs * pl.w * sizeof(float), kWsAlign);
    l.total = off;
    return l;
}

ckv_status check_ws(const Plan& pl, const ckv_batch* b, int T, void* ws, size_t bytes, WsLayout* l) {
    *l = ws_layout(pl, b, T);
    if (!ws) return fail(CKV_ERR_WORKSPACE, "workspace is NULL");
    if (!aligned(ws, kWsAlign)) return fail(CKV_ERR_WORKSPACE, "workspace not 256-byte aligned");
    if (bytes < l->total)
        return fail(CKV_ERR_WORKSPACE, "workspace %zu bytes < required %zu", bytes, l->total);
    return CKV_OK;
}

ckv_status check_kv(const void* p, const char* name, int T) {
    if (T == 0) return CKV_OK;
    if (!p) return fail(CKV_ERR_INVALID_ARG, "%s is NULL", name);
    if (!aligned(p, 16)) return fail(CKV_ERR_INVALID_ARG, "%s is not 16-byte aligned", name);
    return CKV_OK;
}

ckv_status resolve_strides(const Plan& pl, int64_t* tok, int64_t* head) {
    if (*tok == 0) *tok = static_cast<int64_t>(pl.Hkv) * kHeadDim;
    if (*head == 0) *head = kHeadDim;
    if (*tok < 0 || *head < 0 || *tok % 8 || *head % 8)
        return fail(CKV_ERR_INVALID_ARG, "strides must be non-negative multiples of 8 elements");
    if (*tok >= (static_cast<int64_t>(1) << 38) || *head >= (static_cast<int64_t>(1) << 38))
        return fail(CKV_ERR_UNSUPPORTED, "stride too large");
    return CKV_OK;
}

typedef CUresult (*EncodeTiledFn)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*,
                                  const cuuint64_t*, const cuuint64_t*, const cuuint32_t*,
                                  const cuuint32_t*, CUtensorMapInterleave, CUtensorMapSwizzle,
                                  CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

EncodeTiledFn encode_fn() {
    static EncodeTiledFn fn = nullptr;
    if (!fn) {
        void* ptr = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &ptr, 12000, cudaEnableDefault,
                                             &q) == cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            fn = reinterpret_cast<EncodeTiledFn>(ptr);
    }
    return fn;
}

// K viewed as {128 (dim), H_kv, T} with a {64, 1, 128} box and the 128-byte swizzle.
// The window queries [S, w, H_q, 128] as {128 (dim), H_q, S*w (row)}: one box is 64 dims of
// rows_per_box consecutive window rows of one head, 128-byte swizzled like the MMA operand.
ckv_status make_q_map(CUtensorMap* map, const void* q, int Hq, int S, int w, int rows_per_box) {
    EncodeTiledFn fn = encode_fn();
    if (!fn) return fail(CKV_ERR_CUDA, "cuTensorMapEncodeTiled is unavailable");
    const cuuint64_t dims[3] = {static_cast<cuuint64_t>(kHeadDim), static_cast<cuuint64_t>(Hq),
                                static_cast<cuuint64_t>(S) * static_cast<cuuint64_t>(w)};
    const cuuint64_t strides[2] = {static_cast<cuuint64_t>(kHeadDim) * 2,
                                   static_cast<cuuint64_t>(Hq) * kHeadDim * 2};
    const cuuint32_t box[3] = {64, 1, static_cast<cuuint32_t>(rows_per_box)};
    const cuuint32_t estr[3] = {1, 1, 1};
    const CUresult r = fn(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(q), dims,
                          strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE,
                          CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                          CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    if (r != CUDA_SUCCESS) return fail(CKV_ERR_CUDA, "cuTensorMapEncodeTiled failed (%d)", static_cast<int>(r));
    return CKV_OK;
}

ckv_status make_k_map(CUtensorMap* map, const void* k, int Hkv, int T, int64_t tok, int64_t head) {
    EncodeTiledFn fn = encode_fn();
    if (!fn) return fail(CKV_ERR_CUDA, "cuTensorMapEncodeTiled is unavailable");
    const cuuint64_t dims[3] = {static_cast<cuuint64_t>(kHeadDim), static_cast<cuuint64_t>(Hkv),
                                static_cast<cuuint64_t>(T)};
    const cuuint64_t strides[2] = {static_cast<cuuint64_t>(head) * 2, static_cast<cuuint64_t>(tok) * 2};
    const cuuint32_t box[3] = {64, 1, static_cast<cuuint32_t>(kTileKeys)};
    const cuuint32_t estr[3] = {1, 1, 1};
    const CUresult r = fn(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(k), dims,
                          strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE,
                          CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                          CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    if (r != CUDA_SUCCESS) return fail(CKV_ERR_CUDA, "cuTensorMapEncodeTiled failed (%d)", static_cast<int>(r));
    return CKV_OK;
}

// A [n_sel, T] fp32 score buffer as 16-float lines {16, score_map_lines}, a box of
// kScoreMapBoxLines lines, 64-byte swizzled (the multi-layer selection's TMA stage).  The last
// line may run up to 60 bytes past the buffer: its owner keeps 64 bytes of padding there.
ckv_status make_score_map(CUtensorMap* map, const float* scores, int n_sel, int T) {
    EncodeTiledFn fn = encode_fn();
    if (!fn) return fail(CKV_ERR_CUDA, "cuTensorMapEncodeTiled is unavailable");
    const cuuint64_t dims[2] = {16, static_cast<cuuint64_t>(score_map_lines(n_sel, T))};
    const cuuint64_t strides[1] = {64};
    const cuuint32_t box[2] = {16, static_cast<cuuint32_t>(kScoreMapBoxLines)};
    const cuuint32_t estr[2] = {1, 1};
    const CUresult r = fn(map, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 2, const_cast<float*>(scores), dims, strides,
                          box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_64B,
                          CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    if (r != CUDA_SUCCESS) return fail(CKV_ERR_CUDA, "cuTensorMapEncodeTiled failed (%d)", static_cast<int>(r));
    return CKV_OK;
}

}  // namespace

int device_sm_count() {
    static int cached[64] = {0};
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0) return 0;
    if (dev < 64 && cached[dev]) return cached[dev];
    int n = 0;
    if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess) return 0;
    if (dev < 64) cached[dev] = n;
    return n;
}

namespace {

// ---------------------------------------------------------------- two-pass scoring (reload)
// One layer of a scoring call on the two-pass kernel of score_layers.cu.
struct LayerJob {
    const Plan* pl;
    const void* q_win;
    const void* k;
    int64_t tok, head;
    float* scores;
    const float* lse = nullptr;  // the window rows' lse: the single-pass kernel (all jobs or none)
    int64_t lse_stride = 0;
};

// The items of one launch of the two-pass kernel: unit (lb, s), of tiles[s] key tiles, is
// split into m = ceil(tiles / c) items of balanced length, unit after unit (head batch major);
// `units` ends with an entry holding the total.  c is kItemTiles, or more where a unit would
// otherwise have more items than the launch has CTAs (the kernel's progress argument needs at
// most G).  Items are long enough that their fixed costs (taking the item, loading its query
// rows, publishing its sums, computing the unit's lse) are paid rarely, and short enough that
// the faster SMs take more of the work and that the tiles pass 2 re-reads stay in L2.
constexpr int kItemTiles = 14;
void plan_items(const std::vector<int>& tiles, int n_lb, int G, std::vector<LaunchUnit>& units) {
    units.clear();
    int max_tiles = 0;
    for (int t : tiles) max_tiles = std::max(max_tiles, t);
    const int c = std::max(kItemTiles, (max_tiles + G - 1) / G);
    int item = 0;
    for (int lb = 0; lb < n_lb; ++lb)
        for (int s = 0; s < static_cast<int>(tiles.size()); ++s) {
            const int t = tiles[s];
            if (t == 0) continue;
            units.push_back(LaunchUnit{static_cast<int16_t>(lb), static_cast<int16_t>(s), item});
            item += std::min(t, (t + c - 1) / c);
        }
    units.push_back(LaunchUnit{0, 0, item});
}

// Sequences per launch of the two-pass kernel when a layer has up to max_nb head batches: one
// layer's units of one chunk always fit a launch's unit table.
int launch_seq_chunk(int max_nb) {
    return std::max(1, std::min(kMaxLaunchSeqs, kMaxLaunchUnits / std::max(1, max_nb)));
}

// Enqueues the scoring of `jobs` (layers sharing the batch and the window) on the two-pass
// kernel, or on the single-pass one where the jobs carry their lse: one persistent launch per
// chunk of sequences (launch_seq_chunk) and per group of consecutive layers whose tables fit
// the kernel's parameters.  Sequences of at most skip_le tokens are skipped.  `sums`/`counters`
// hold the exchange of every unit of one launch and its item counter (each launch clears them
// first; launches are ordered on `stream`).
ckv_status enqueue_layers(const std::vector<LayerJob>& jobs, const ckv_batch* b, int T, void* sums,
                          int* counters, int* status, int skip_le, int max_ctas, cudaStream_t stream) {
    if (jobs.empty()) return CKV_OK;
    int ctas = device_sm_count();
    if (ctas <= 0) return cuda_fail(cudaGetLastError(), "querying the SM count");
    if (max_ctas > 0) ctas = std::min(ctas, max_ctas);
    const int S = b->num_seqs;
    const int w_pad = jobs[0].pl->w_pad, w = jobs[0].pl->w;
    static thread_local LayersLaunch L;
    const uint32_t hash = seqlens_hash(b->cu_seqlens_host, S);
    std::vector<int> tiles;
    int max_nb = 1;
    for (const LayerJob& J : jobs) max_nb = std::max(max_nb, J.pl->nb);
    const int chunk = launch_seq_chunk(max_nb);
    for (int s0 = 0; s0 < S; s0 += chunk) {  // chunks of sequences
        const int s1 = std::min(S, s0 + chunk);
        tiles.clear();
        L.seq_start.clear();
        L.seq_len.clear();
        int active = 0;
        for (int s = s0; s < s1; ++s) {
            const int len = b->cu_seqlens_host[s + 1] - b->cu_seqlens_host[s];
            const int t = len > skip_le && len > 0 ? (len + kTileKeys - 1) / kTileKeys : 0;
            if (t > 32767) return fail(CKV_ERR_UNSUPPORTED, "a sequence of more than 2^22 tokens");
            tiles.push_back(t);
            active += t > 0;
            L.seq_start.push_back(b->cu_seqlens_host[s]);
            L.seq_len.push_back(len);
        }
        if (active == 0) continue;
        size_t j0 = 0;
        while (j0 < jobs.size()) {
            // the layers of this launch: as many as the parameter tables hold
            size_t j1 = j0;
            int nb = 0, nsel = 0, n_cols = 32;
            while (j1 < jobs.size() && static_cast<int>(j1 - j0) < kMaxLaunchLayers &&
                   nb + jobs[j1].pl->nb <= kMaxLaunchBatches &&
                   nsel + jobs[j1].pl->n_sel <= kMaxLaunchSel &&
                   (nb + jobs[j1].pl->nb) * active <= kMaxLaunchUnits) {
                nb += jobs[j1].pl->nb;
                nsel += jobs[j1].pl->n_sel;
                n_cols = std::max(n_cols, jobs[j1].pl->n_cols);
                ++j1;
            }
            if (j1 == j0)
                return fail(CKV_ERR_UNSUPPORTED, "a layer's head batches and sequences exceed one launch's tables");
            L.layers.clear();
            L.batch_layer.clear();
            L.batch_group.clear();
            L.batch_first.clear();
            L.batch_nheads.clear();
            L.batch_sel.clear();
            L.sel_heads.clear();
            for (size_t j = j0; j < j1; ++j) {
                const LayerJob& J = jobs[j];
                LayersLayer ly;
                ckv_status st;
                if ((st = make_k_map(&ly.tmap_k, J.k, J.pl->Hkv, T, J.tok, J.head))) return st;
                if ((st = make_q_map(&ly.tmap_q, J.q_win, J.pl->Hq, S, w, w_pad))) return st;
                ly.scores = J.scores;
                ly.lse = J.lse;
                ly.lse_stride = J.lse_stride;
                const int sel_base = static_cast<int>(L.sel_heads.size());
                for (int bt = 0; bt < J.pl->nb; ++bt) {
                    L.batch_layer.push_back(static_cast<int16_t>(j - j0));
                    L.batch_group.push_back(static_cast<int16_t>(J.pl->batch_group[bt]));
                    L.batch_first.push_back(static_cast<int16_t>(J.pl->batch_first[bt]));
                    L.batch_nheads.push_back(static_cast<int16_t>(J.pl->batch_nheads[bt]));
                    L.batch_sel.push_back(static_cast<int16_t>(sel_base + J.pl->batch_first[bt]));
                }
                for (int h : J.pl->sel_heads) L.sel_heads.push_back(static_cast<int16_t>(h));
                L.layers.push_back(ly);
            }
            plan_items(tiles, nb, ctas, L.units);
            L.seq0 = s0;
            L.S_all = S;
            L.cu_seqlens_dev = b->cu_seqlens_dev;
            L.sums = static_cast<double*>(sums);
            L.counters = counters;
            L.status = status;
            L.T = T;
            L.w = w;
            L.w_pad = w_pad;
            L.n_cols = n_cols;
            L.grid = ctas;
            L.cu_hash = hash;
            L.softmax_scale = jobs[j0].pl->scale;
            L.given_lse = jobs[j0].lse != nullptr;
            const cudaError_t e = launch_score_layers(L, stream);
            if (e != cudaSuccess) return cuda_fail(e, "launching the two-pass scoring kernel");
            j0 = j1;
        }
    }
    return CKV_OK;
}

// Whether the single-layer scoring runs on the TMEM-resident kernel (score_resident.cu); the
// two-pass reload kernel otherwise.  CKV_ERR_UNSUPPORTED when the caller asked for the resident
// kernel and a sequence does not fit it.
ckv_status resident_choice(const Plan& pl, const ckv_batch* b, int skip_le, int ctas, bool* resident) {
    int max_tiles = 0;
    for (int s = 0; s < b->num_seqs; ++s) {
        const int len = b->cu_seqlens_host[s + 1] - b->cu_seqlens_host[s];
        if (len > skip_le && len > 0) max_tiles = std::max(max_tiles, (len + kTileKeys - 1) / kTileKeys);
    }
    const int c_res = 512 / pl.n_cols;
    const bool fits = static_cast<long long>(max_tiles) <= static_cast<long long>(c_res) * ctas;
    if (pl.score_path == CKV_SCORE_RESIDENT && !fits)
        return fail(CKV_ERR_UNSUPPORTED,
                    "resident scoring: a sequence of %d key tiles needs items of at most %d tiles "
                    "on at least %d CTAs (%d available)", max_tiles, c_res,
                    (max_tiles + c_res - 1) / c_res, ctas);
    *resident = fits && (pl.score_path == CKV_SCORE_RESIDENT ||
                         (pl.score_path == CKV_SCORE_AUTO && pl.n_cols == 32));
    return CKV_OK;
}

ckv_status enqueue_score(const Plan& pl, const ckv_batch* b, int T, const void* q_win,
                         const void* k, int64_t tok, int64_t head, float* scores, void* ws,
                         const WsLayout& l, int skip_le, cudaStream_t stream,
                         int max_items_per_launch = kMaxScoreItems, const float* lse = nullptr,
                         int64_t lse_head_stride = 0) {
    int ctas = device_sm_count();
    if (ctas <= 0) return cuda_fail(cudaGetLastError(), "querying the SM count");
    if (pl.max_ctas > 0) ctas = std::min(ctas, pl.max_ctas);
    if (!lse) {
        bool resident = false;
        ckv_status st = resident_choice(pl, b, skip_le, std::min(ctas, max_items_per_launch), &resident);
        if (st) return st;
        if (!resident) {  // the two-pass kernel
            uint8_t* w8 = static_cast<uint8_t*>(ws);
            const std::vector<LayerJob> jobs{LayerJob{&pl, q_win, k, tok, head, scores}};
            return enqueue_layers(jobs, b, T, w8 + l.sums, reinterpret_cast<int*>(w8 + l.unit_counters),
                                  reinterpret_cast<int*>(w8), skip_le, ctas, stream);
        }
    }
    static thread_local ScoreLaunch L;  // reused: keeps the plan's vectors allocated
    ckv_status st = lse ? plan_score_stream(pl, b, skip_le, std::min(ctas, max_items_per_launch), L,
                                            max_items_per_launch)
                        : plan_score(pl, b, skip_le, std::min(ctas, max_items_per_launch), L,
                                     max_items_per_launch);
    if (st) return st;
    L.lse = lse;
    L.lse_head_stride = lse_head_stride;
    if (L.slices.empty()) return CKV_OK;
    if ((st = make_k_map(&L.tmap_k, k, pl.Hkv, T, tok, head))) return st;
    if ((st = make_q_map(&L.tmap_q, q_win, pl.Hq, b->num_seqs, pl.w, pl.w_pad))) return st;
    uint8_t* w8 = static_cast<uint8_t*>(ws);
    L.q_win = q_win;
    L.cu_seqlens_dev = b->cu_seqlens_dev;
    L.partials = w8 + l.partials;
    L.counters = reinterpret_cast<int*>(w8 + l.counters);
    L.scores = scores;
    L.status = reinterpret_cast<int*>(w8);
    L.S = b->num_seqs;
    L.T = T;
    L.Hq = pl.Hq;
    L.w = pl.w;
    L.w_pad = pl.w_pad;
    L.n_cols = pl.n_cols;
    L.nb = pl.nb;
    L.cu_hash = seqlens_hash(b->cu_seqlens_host, b->num_seqs);
    L.softmax_scale = pl.scale;
    L.n_sel = pl.n_sel;
    L.batch_group = pl.batch_group.data();
    L.batch_first = pl.batch_first.data();
    L.batch_nheads = pl.batch_nheads.data();
    L.sel_heads = pl.sel_heads.data();
    const cudaError_t e = launch_score(L, stream);
    if (e != cudaSuccess) return cuda_fail(e, "launching the scoring kernel");
    return CKV_OK;
}

SelectLaunch select_launch(const Plan& pl, const ckv_batch* b, int T, int T_keep, int skip_le,
                           const ckv_config* cfg, void* ws, const WsLayout* l) {
    SelectLaunch L;
    memset(&L, 0, sizeof L);
    if (l) {
        uint8_t* w8 = static_cast<uint8_t*>(ws);
        L.hist = reinterpret_cast<int*>(w8 + l->hist);
        L.arrivals = reinterpret_cast<int*>(w8 + l->arrivals);
        L.chunk_start = reinterpret_cast<int*>(w8 + l->chunk_start);
        L.buckets = w8 + l->buckets;
        L.info = reinterpret_cast<int*>(w8 + l->info);
        L.chunk_off = reinterpret_cast<int*>(w8 + l->chunk_off);
        L.max_chunks = l->max_chunks;
    }
    L.cu_seqlens_dev = b->cu_seqlens_dev;
    L.status = static_cast<int*>(ws);
    L.S = b->num_seqs;
    L.T = T;
    L.Hkv = pl.Hkv;
    L.w = pl.w;
    L.budget = pl.budget;
    L.T_keep = T_keep;
    L.pool_kernel = cfg->pool_kernel;
    L.pool_type = cfg->pool_type;
    L.head_order = cfg->head_order;
    L.skip_le = skip_le;
    L.cu_hash = seqlens_hash(b->cu_seqlens_host, b->num_seqs);
    L.group_first = pl.group_first.data();
    L.n_vec = pl.n_vec;
    L.min_len = INT_MAX;
    L.max_len = 0;
    for (int s = 0; s < b->num_seqs; ++s) {
        const int len = b->cu_seqlens_host[s + 1] - b->cu_seqlens_host[s];
        L.min_len = std::min(L.min_len, len);
        L.max_len = std::max(L.max_len, len);
    }
    return L;
}

}  // namespace

// Limit of the kernels' bounded waits on other roles and other CTAs (ckv_set_wait_limit_us).
std::atomic<long long> g_wait_cycles{kWaitTimeoutCycles};

long long wait_limit_cycles() { return g_wait_cycles.load(std::memory_order_relaxed); }

// The last-error message for the other translation units (host-only entry points).
ckv_status set_error(ckv_status st, const char* fmt, ...) {
    va_list ap;
    va_start(ap, fmt);
    vsnprintf(g_msg, sizeof g_msg, fmt, ap);
    va_end(ap);
    return st;
}
}  // namespace ckv

using namespace ckv;

extern "C" {

int32_t ckv_abi_version(void) { return CKV_ABI_VERSION; }

ckv_status ckv_set_wait_limit_us(uint32_t microseconds) {
    long long cycles = kWaitTimeoutCycles;
    if (microseconds > 0) {
        int khz = 0;  // SM clock; 2 GHz if there is no device to ask
        int dev = 0;
        if (cudaGetDevice(&dev) != cudaSuccess ||
            cudaDeviceGetAttribute(&khz, cudaDevAttrClockRate, dev) != cudaSuccess || khz <= 0) {
            cudaGetLastError();
            khz = 2000000;
        }
        cycles = static_cast<long long>(microseconds) * khz / 1000;
        if (cycles < 1) cycles = 1;
    }
    g_wait_cycles.store(cycles, std::memory_order_relaxed);
    return CKV_OK;
}

const char* ckv_status_string(ckv_status s) {
    switch (s) {
        case CKV_OK: return "CKV_OK";
        case CKV_ERR_INVALID_ARG: return "CKV_ERR_INVALID_ARG";
        case CKV_ERR_UNSUPPORTED: return "CKV_ERR_UNSUPPORTED";
        case CKV_ERR_WORKSPACE: return "CKV_ERR_WORKSPACE";
        case CKV_ERR_CUDA: return "CKV_ERR_CUDA";
        case CKV_ERR_DEVICE: return "CKV_ERR_DEVICE";
    }
    return "unknown ckv_status";
}

const char* ckv_last_error_message(void) { return g_msg; }

ckv_status ckv_workspace_size(const ckv_config* cfg, int32_t layer, const ckv_batch* batch,
                              size_t* bytes) {
    Plan pl;
    ckv_status st = make_plan(cfg, layer, pl);
    if (st) return st;
    int T = 0;
    if ((st = check_batch(batch, &T))) return st;
    if (!bytes) return fail(CKV_ERR_INVALID_ARG, "bytes is NULL");
    *bytes = ws_layout(pl, batch, T).total;
    return CKV_OK;
}

ckv_status ckv_keep_lengths(const ckv_config* cfg, int32_t layer, const ckv_batch* batch,
                            int32_t* cu_keep_host, int32_t* n_sel) {
    Plan pl;
    ckv_status st = make_plan(cfg, layer, pl);
    if (st) return st;
    int T = 0;
    if ((st = check_batch(batch, &T))) return st;
    if (!cu_keep_host) return fail(CKV_ERR_INVALID_ARG, "cu_keep_host is NULL");
    cu_keep_host[0] = 0;
    for (int s = 0; s < batch->num_seqs; ++s)
        cu_keep_host[s + 1] = cu_keep_host[s] +
                              std::min(pl.budget, batch->cu_seqlens_host[s + 1] - batch->cu_seqlens_host[s]);
    if (n_sel) *n_sel = pl.n_sel;
    return CKV_OK;
}

}  // extern "C"

namespace {

// The given lse array: device, 4-byte aligned, [H_q][lse_head_stride] with lse_head_stride >= S*w
// (0 selects S*w).
ckv_status check_lse(const Plan& pl, const ckv_batch* b, const float* lse, int64_t* stride) {
    if (!lse) return fail(CKV_ERR_INVALID_ARG, "lse is NULL");
    if (!aligned(lse, 4)) return fail(CKV_ERR_INVALID_ARG, "lse is not 4-byte aligned");
    const int64_t rows = static_cast<int64_t>(b->num_seqs) * pl.w;
    if (*stride == 0) *stride = rows;
    if (*stride < rows) return fail(CKV_ERR_INVALID_ARG, "lse_head_stride %lld < S*w", (long long)*stride);
    return CKV_OK;
}

ckv_status score_window_impl(const ckv_config* cfg, int32_t layer, const ckv_batch* batch,
                             const void* q_win, const void* k, int64_t tok_stride,
                             int64_t head_stride, const float* lse, int64_t lse_head_stride,
                             float* scores, void* workspace, size_t workspace_bytes,
                             ckv_stream stream) {
    Plan pl;
    ckv_status st = make_plan(cfg, layer, pl);
    if (st) return st;
    int T = 0;
    WsLayout l;
    if ((st = check_batch(batch, &T)) || (st = resolve_strides(pl, &tok_stride, &head_stride)) ||
        (st = check_kv(q_win, "q_win", T)) || (st = check_kv(k, "k", T)) ||
        (st = check_kv(scores, "scores", T)) ||
        (st = check_ws(pl, batch, T, workspace, workspace_bytes, &l)))
        return st;
    if (lse && (st = check_lse(pl, batch, lse, &lse_head_stride))) return st;
    return enqueue_score(pl, batch, T, q_win, k, tok_stride, head_stride, scores, workspace, l, -1,
                         reinterpret_cast<cudaStream_t>(stream), kMaxScoreItems, lse, lse_head_stride);
}

}  // namespace

extern "C" {

ckv_status ckv_score_window(const ckv_config* cfg, int32_t layer, const ckv_batch* batch,
                            const void* q_win, const void* k, int64_t tok_stride,
                            int64_t head_stride, float* scores, void* workspace,
                            size_t workspace_bytes, ckv_stream stream) {
    return score_window_impl(cfg, layer, batch, q_win, k, tok_stride, head_stride, nullptr, 0,
                             scores, workspace, workspace_bytes, stream);
}

ckv_status ckv_score_window_lse(const ckv_config* cfg, int32_t layer, const ckv_batch* batch,
                                const void* q_win, const void* k, int64_t tok_stride,
                                int64_t head_stride, const float* lse, int64_t lse_head_stride,
                                float* scores, void* workspace, size_t workspace_bytes,
                                ckv_stream stream) {
    if (!lse) return fail(CKV_ERR_INVALID_ARG, "lse is NULL");
    return score_window_impl(cfg, layer, batch, q_win, k, tok_stride, head_stride, lse,
                             lse_head_stride, scores, workspace, workspace_bytes, stream);
}

ckv_status ckv_pool(const ckv_config* cfg, int32_t layer, const ckv_batch* batch,
                    const float* scores, float* pooled, ckv_stream stream) {
    Plan pl;
    ckv_status st = make_plan(cfg, layer, pl);
    if (st) return st;
    int T = 0;
    if ((st = check_batch(batch, &T)) || (st = check_kv(scores, "scores", T)) ||
        (st = check_kv(pooled, "pooled", T)))
        return st;
    SelectLaunch L = select_launch(pl, batch, T, 0, -1, cfg, nullptr, nullptr);
    L.scores = scores;
    L.pooled = pooled;
    const cudaError_t e = launch_pool(L, reinterpret_cast<cudaStream_t>(stream));
    return e == cudaSuccess ? CKV_OK : cuda_fail(e, "launching the pooling kernel");
}

ckv_status ckv_select_topk(const ckv_config* cfg, int32_t layer, const ckv_batch* batch,
                           const float* pooled, int32_t* idx, int32_t* cu_keep_dev,
                           void* workspace, size_t workspace_bytes, ckv_stream stream) {
    Plan pl;
    ckv_status st = make_plan(cfg, layer, pl);
    if (st) return st;
    int T = 0;
    WsLayout l;
    if ((st = check_batch(batch, &T)) || (st = check_kv(pooled, "pooled", T)) ||
        (st = check_ws(pl, batch, T, workspace, workspace_bytes, &l)))
        return st;
    const int64_t tk = keep_total(batch, pl.budget);
    if (tk > 0 && !idx) return fail(CKV_ERR_INVALID_ARG, "idx is NULL");
    if (!cu_keep_dev) return fail(CKV_ERR_INVALID_ARG, "cu_keep_dev is NULL");
    SelectLaunch L = select_launch(pl, batch, T, static_cast<int>(tk), -1, cfg, workspace, &l);
    L.pooled = const_cast<float*>(pooled);
    L.idx = idx;
    L.cu_keep_dev = cu_keep_dev;
    L.from_scores = 0;
    L.write_pooled = 0;
    const cudaError_t e = launch_select(L, reinterpret_cast<cudaStream_t>(stream));
    return e == cudaSuccess ? CKV_OK : cuda_fail(e, "launching the selection kernel");
}

ckv_status ckv_gather_compact(const ckv_config* cfg, const ckv_batch* batch, int32_t t_keep,
                              const void* k, const void* v, int64_t tok_stride,
                              int64_t head_stride, const int32_t* idx,
                              const int32_t* cu_keep_dev, void* k_out, void* v_out,
                              void* workspace, size_t workspace_bytes, ckv_stream stream) {
    ckv_status st = check_config(cfg);
    if (st) return st;
    Plan pl;
    pl.Hkv = cfg->num_kv_heads;
    int T = 0;
    if ((st = check_batch(batch, &T)) || (st = resolve_strides(pl, &tok_stride, &head_stride)))
        return st;
    if (!workspace || !aligned(workspace, kWsAlign) || workspace_bytes < sizeof(WsHeader))
        return fail(CKV_ERR_WORKSPACE, "workspace missing, misaligned or too small");
    if (t_keep < 0) return fail(CKV_ERR_INVALID_ARG, "t_keep %d < 0", t_keep);
    if (t_keep == 0) return CKV_OK;
    if ((st = check_kv(k, "k", T)) || (st = check_kv(v, "v", T)) ||
        (st = check_kv(k_out, "k_out", t_keep)) || (st = check_kv(v_out, "v_out", t_keep)))
        return st;
    if (!idx || !cu_keep_dev) return fail(CKV_ERR_INVALID_ARG, "idx and cu_keep_dev are required");
    GatherLaunch L;
    L.k = k;
    L.v = v;
    L.tok_stride = tok_stride;
    L.head_stride = head_stride;
    L.idx = idx;
    L.cu_keep_dev = cu_keep_dev;
    L.cu_seqlens_dev = batch->cu_seqlens_dev;
    L.k_out = k_out;
    L.v_out = v_out;
    L.status = static_cast<int*>(workspace);
    L.S = batch->num_seqs;
    L.T = T;
    L.Hkv = pl.Hkv;
    L.T_keep = t_keep;
    L.cu_hash = seqlens_hash(batch->cu_seqlens_host, batch->num_seqs);
    const cudaError_t e = launch_gather(L, reinterpret_cast<cudaStream_t>(stream));
    return e == cudaSuccess ? CKV_OK : cuda_fail(e, "launching the gather kernel");
}

}  // extern "C"

namespace {

// The fused selection (pool, top-k, compaction, gather) of one layer from `scores`.
ckv_status enqueue_select_fused(const Plan& pl, const ckv_config* cfg, const ckv_batch* batch, int T,
                                const float* scores, const void* k, const void* v,
                                int64_t tok_stride, int64_t head_stride, int32_t* idx,
                                int32_t* cu_keep_dev, void* k_out, void* v_out, float* pooled_out,
                                void* workspace, WsLayout& l, int64_t tk, cudaStream_t s) {
    uint8_t* w8 = static_cast<uint8_t*>(workspace);
    float* pooled = pooled_out ? pooled_out : reinterpret_cast<float*>(w8 + l.pooled);
    const int skip_le = pl.budget;  // sequences that fit the budget are kept whole
    SelectLaunch L = select_launch(pl, batch, T, static_cast<int>(tk), skip_le, cfg, workspace, &l);
    L.scores = const_cast<float*>(scores);
    L.pooled = pooled;
    L.idx = idx;
    L.cu_keep_dev = cu_keep_dev;
    L.from_scores = 1;                      // pooling is fused into the selection
    L.write_pooled = pooled_out != nullptr;
    if (tk > 0) {                           // and so is the gather
        L.k = k;
        L.v = v;
        L.tok_stride = tok_stride;
        L.head_stride = head_stride;
        L.k_out = k_out;
        L.v_out = v_out;
    }
    const cudaError_t e = launch_select(L, s);
    return e == cudaSuccess ? CKV_OK : cuda_fail(e, "launching the pool, selection and gather kernels");
}

// Checks of the selection's outputs, shared by the fused calls; *tk_out = kept tokens.
ckv_status check_select_outputs(const ckv_batch* batch, const Plan& pl, int32_t* idx,
                                int32_t* cu_keep_dev, void* k_out, void* v_out, float* pooled_out,
                                int64_t* tk_out) {
    ckv_status st;
    if (pooled_out && !aligned(pooled_out, 16))
        return fail(CKV_ERR_INVALID_ARG, "pooled_out is not 16-byte aligned");
    const int64_t tk = keep_total(batch, pl.budget);
    if (tk > INT32_MAX) return fail(CKV_ERR_UNSUPPORTED, "too many kept tokens");
    if (!cu_keep_dev) return fail(CKV_ERR_INVALID_ARG, "cu_keep_dev is NULL");
    if (tk > 0 && (st = check_kv(idx, "idx", 1))) return st;
    if (tk > 0 && ((st = check_kv(k_out, "k_out", 1)) || (st = check_kv(v_out, "v_out", 1))))
        return st;
    *tk_out = tk;
    return CKV_OK;
}

ckv_status compress_layer_impl(const ckv_config* cfg, int32_t layer, const ckv_batch* batch,
                               const void* q_win, const void* k, const void* v,
                               int64_t tok_stride, int64_t head_stride, const float* lse,
                               int64_t lse_head_stride, int32_t* idx, int32_t* cu_keep_dev,
                               void* k_out, void* v_out, float* pooled_out, void* workspace,
                               size_t workspace_bytes, ckv_stream stream) {
    Plan pl;
    ckv_status st = make_plan(cfg, layer, pl);
    if (st) return st;
    int T = 0;
    WsLayout l;
    if ((st = check_batch(batch, &T)) || (st = resolve_strides(pl, &tok_stride, &head_stride)) ||
        (st = check_kv(q_win, "q_win", T)) || (st = check_kv(k, "k", T)) ||
        (st = check_kv(v, "v", T)) || (st = check_ws(pl, batch, T, workspace, workspace_bytes, &l)))
        return st;
    if (lse && (st = check_lse(pl, batch, lse, &lse_head_stride))) return st;
    int64_t tk = 0;
    if ((st = check_select_outputs(batch, pl, idx, cu_keep_dev, k_out, v_out, pooled_out, &tk)))
        return st;
    cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
    float* scores = reinterpret_cast<float*>(static_cast<uint8_t*>(workspace) + l.scores);
    const int skip_le = pl.budget;  // sequences that fit the budget are kept whole
    if ((st = enqueue_score(pl, batch, T, q_win, k, tok_stride, head_stride, scores, workspace, l,
                            skip_le, s, kMaxScoreItems, lse, lse_head_stride)))
        return st;
    return enqueue_select_fused(pl, cfg, batch, T, scores, k, v, tok_stride, head_stride, idx,
                                cu_keep_dev, k_out, v_out, pooled_out, workspace, l, tk, s);
}

}  // namespace

extern "C" {

ckv_status ckv_select_compact(const ckv_config* cfg, int32_t layer, const ckv_batch* batch,
                              const float* scores, const void* k, const void* v,
                              int64_t tok_stride, int64_t head_stride, int32_t* idx,
                              int32_t* cu_keep_dev, void* k_out, void* v_out, float* pooled_out,
                              void* workspace, size_t workspace_bytes, ckv_stream stream) {
    Plan pl;
    ckv_status st = make_plan(cfg, layer, pl);
    if (st) return st;
    int T = 0;
    WsLayout l;
    if ((st = check_batch(batch, &T)) || (st = resolve_strides(pl, &tok_stride, &head_stride)) ||
        (st = check_kv(k, "k", T)) || (st = check_kv(v, "v", T)) ||
        (st = check_ws(pl, batch, T, workspace, workspace_bytes, &l)))
        return st;
    if (!scores) return fail(CKV_ERR_INVALID_ARG, "scores is NULL");
    if (!aligned(scores, 16)) return fail(CKV_ERR_INVALID_ARG, "scores is not 16-byte aligned");
    int64_t tk = 0;
    if ((st = check_select_outputs(batch, pl, idx, cu_keep_dev, k_out, v_out, pooled_out, &tk)))
        return st;
    return enqueue_select_fused(pl, cfg, batch, T, scores, k, v, tok_stride, head_stride, idx,
                                cu_keep_dev, k_out, v_out, pooled_out, workspace, l, tk,
                                reinterpret_cast<cudaStream_t>(stream));
}

ckv_status ckv_compress_layer(const ckv_config* cfg, int32_t layer, const ckv_batch* batch,
                              const void* q_win, const void* k, const void* v,
                              int64_t tok_stride, int64_t head_stride, int32_t* idx,
                              int32_t* cu_keep_dev, void* k_out, void* v_out, float* pooled_out,
                              void* workspace, size_t workspace_bytes, ckv_stream stream) {
    return compress_layer_impl(cfg, layer, batch, q_win, k, v, tok_stride, head_stride, nullptr, 0,
                               idx, cu_keep_dev, k_out, v_out, pooled_out, workspace,
                               workspace_bytes, stream);
}

ckv_status ckv_compress_layer_lse(const ckv_config* cfg, int32_t layer, const ckv_batch* batch,
                                  const void* q_win, const void* k, const void* v,
                                  int64_t tok_stride, int64_t head_stride, const float* lse,
                                  int64_t lse_head_stride, int32_t* idx, int32_t* cu_keep_dev,
                                  void* k_out, void* v_out, float* pooled_out, void* workspace,
                                  size_t workspace_bytes, ckv_stream stream) {
    if (!lse) return fail(CKV_ERR_INVALID_ARG, "lse is NULL");
    return compress_layer_impl(cfg, layer, batch, q_win, k, v, tok_stride, head_stride, lse,
                               lse_head_stride, idx, cu_keep_dev, k_out, v_out, pooled_out,
                               workspace, workspace_bytes, stream);
}

}  // extern "C"

namespace {

// Workspace of a multi-layer call: the header and one layer's selection scratch (the layout of
// the layer needing the most), the two-pass kernel's exchange for every (head batch, sequence)
// unit of the call's layers, then each layer's scores (ckv_compress_layers).
struct LayersWs {
    WsLayout sel;
    size_t sums = 0, counters = 0, next_unit = 0, total = 0;
    std::vector<size_t> scores, keys;  // per layer (ckv_compress_layers)
};

ckv_status prepare_layers(const ckv_config* cfg, int32_t n_layers, const ckv_layer_io* io,
                          const ckv_batch* b, std::vector<Plan>& pls, int* T, LayersWs* lw) {
    ckv_status st;
    if (n_layers < 1) return fail(CKV_ERR_INVALID_ARG, "n_layers %d < 1", n_layers);
    if (!io) return fail(CKV_ERR_INVALID_ARG, "io is NULL");
    if ((st = check_batch(b, T))) return st;
    pls.assign(n_layers, Plan());
    size_t units = 0, best = 0;
    for (int i = 0; i < n_layers; ++i) {
        if ((st = make_plan(cfg, io[i].layer, pls[i]))) return st;
        units += static_cast<size_t>(pls[i].nb) * b->num_seqs;
        const WsLayout l = ws_layout(pls[i], b, *T);
        if (i == 0 || l.total > best) {
            best = l.total;
            lw->sel = l;
        }
    }
    size_t off = round_up(lw->sel.total, kWsAlign);
    lw->sums = off;
    off = round_up(off + units * kMaxCols * sizeof(double), kWsAlign);
    lw->counters = off;  // and, after them, the kernel's item counter
    off = round_up(off + (units + 1) * sizeof(int), kWsAlign);
    lw->next_unit = off;  // the selection kernel's work counter
    off = round_up(off + sizeof(int), kWsAlign);
    lw->scores.assign(n_layers, 0);
    lw->keys.assign(n_layers, 0);
    for (int i = 0; i < n_layers; ++i) {
        lw->scores[i] = off;  // 64 bytes of padding after: the last line of the scores' tensor map
        off = round_up(off + static_cast<size_t>(pls[i].n_sel) * *T * sizeof(float) + 64, kWsAlign);
        lw->keys[i] = off;  // the selection's (key, position) candidates, [H_kv, key stride]
        off = round_up(off + static_cast<size_t>(pls[i].Hkv) * select_key_stride(*T, b->num_seqs) *
                                 2 * sizeof(uint32_t), kWsAlign);
    }
    lw->total = off;
    return CKV_OK;
}

ckv_status check_layers_ws(const LayersWs& lw, void* ws, size_t bytes, bool with_scores) {
    if (!ws) return fail(CKV_ERR_WORKSPACE, "workspace is NULL");
    if (!aligned(ws, kWsAlign)) return fail(CKV_ERR_WORKSPACE, "workspace not 256-byte aligned");
    const size_t need = with_scores ? lw.total : lw.scores.empty() ? lw.total : lw.scores[0];
    if (bytes < need) return fail(CKV_ERR_WORKSPACE, "workspace %zu bytes < required %zu", bytes, need);
    return CKV_OK;
}

// The scoring jobs of a multi-layer call; scores in the workspace when `own_scores`.
ckv_status layer_jobs(const std::vector<Plan>& pls, const ckv_layer_io* io, int T, uint8_t* w8,
                      const LayersWs& lw, bool own_scores, std::vector<LayerJob>& jobs,
                      std::vector<int64_t>& tok, std::vector<int64_t>& head) {
    ckv_status st;
    const int n = static_cast<int>(pls.size());
    jobs.clear();
    tok.assign(n, 0);
    head.assign(n, 0);
    for (int i = 0; i < n; ++i) {
        tok[i] = io[i].tok_stride;
        head[i] = io[i].head_stride;
        if ((st = resolve_strides(pls[i], &tok[i], &head[i])) || (st = check_kv(io[i].q_win, "q_win", T)) ||
            (st = check_kv(io[i].k, "k", T)))
            return st;
        if (pls[i].w != pls[0].w) return fail(CKV_ERR_INVALID_ARG, "layers with different windows");
        float* sc = own_scores ? reinterpret_cast<float*>(w8 + lw.scores[i]) : io[i].scores;
        if (!own_scores && (st = check_kv(sc, "scores", T))) return st;
        jobs.push_back(LayerJob{&pls[i], io[i].q_win, io[i].k, tok[i], head[i], sc});
    }
    return CKV_OK;
}

// Each layer's given lse (io[i].lse, checked as for the one-layer call) into its scoring job.
ckv_status layer_lse(const std::vector<Plan>& pls, const ckv_layer_io* io, const ckv_batch* b,
                     std::vector<LayerJob>& jobs) {
    ckv_status st;
    for (size_t i = 0; i < jobs.size(); ++i) {
        if (!io[i].lse) return fail(CKV_ERR_INVALID_ARG, "io[%zu].lse is NULL", i);
        int64_t stride = io[i].lse_head_stride;
        if ((st = check_lse(pls[i], b, io[i].lse, &stride))) return st;
        jobs[i].lse = io[i].lse;
        jobs[i].lse_stride = stride;
    }
    return CKV_OK;
}

// ckv_compress_layers(_lse): the layers' scoring (one persistent launch, two-pass or, with the
// lse given, single-pass) into the workspace, then every layer's selection in one launch.
ckv_status compress_layers_impl(const ckv_config* cfg, int32_t n_layers, const ckv_layer_io* io,
                                const ckv_batch* batch, void* workspace, size_t workspace_bytes,
                                ckv_stream stream, bool given_lse) {
    static thread_local std::vector<Plan> pls;
    static thread_local std::vector<LayerJob> jobs;
    static thread_local std::vector<int64_t> tok, head;
    LayersWs lw;
    int T = 0;
    ckv_status st;
    if ((st = prepare_layers(cfg, n_layers, io, batch, pls, &T, &lw)) ||
        (st = check_layers_ws(lw, workspace, workspace_bytes, true)))
        return st;
    uint8_t* w8 = static_cast<uint8_t*>(workspace);
    if ((st = layer_jobs(pls, io, T, w8, lw, true, jobs, tok, head))) return st;
    std::vector<int64_t> tks(n_layers, 0);
    int min_budget = INT_MAX;
    for (int i = 0; i < n_layers; ++i) {
        if ((st = check_kv(io[i].v, "v", T)) ||
            (st = check_select_outputs(batch, pls[i], io[i].idx, io[i].cu_keep_dev, io[i].k_out,
                                       io[i].v_out, io[i].pooled_out, &tks[i])))
            return st;
        min_budget = std::min(min_budget, pls[i].budget);
    }
    if (given_lse && (st = layer_lse(pls, io, batch, jobs))) return st;
    cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
    // sequences that fit every layer's budget are kept whole by every selection
    if ((st = enqueue_layers(jobs, batch, T, w8 + lw.sums, reinterpret_cast<int*>(w8 + lw.counters),
                             reinterpret_cast<int*>(w8), min_budget, cfg->max_ctas, s)))
        return st;
    // every layer's selection in one launch (one per 32 layers)
    static thread_local std::vector<SelectLaunch> sls;
    static thread_local std::vector<uint32_t*> keys;
    static thread_local std::vector<CUtensorMap> maps;
    sls.assign(n_layers, SelectLaunch{});
    keys.assign(n_layers, nullptr);
    maps.resize(n_layers);
    for (int i = 0; i < n_layers; ++i) {
        SelectLaunch& L = sls[i];
        L = select_launch(pls[i], batch, T, static_cast<int>(tks[i]), pls[i].budget, cfg, workspace, &lw.sel);
        L.scores = jobs[i].scores;
        if ((st = make_score_map(&maps[i], jobs[i].scores, pls[i].n_sel, T))) return st;
        L.score_map = &maps[i];
        L.pooled = io[i].pooled_out;
        L.write_pooled = io[i].pooled_out != nullptr;
        L.from_scores = 1;
        L.idx = io[i].idx;
        L.cu_keep_dev = io[i].cu_keep_dev;
        if (tks[i] > 0) {
            L.k = io[i].k;
            L.v = io[i].v;
            L.tok_stride = tok[i];
            L.head_stride = head[i];
            L.k_out = io[i].k_out;
            L.v_out = io[i].v_out;
        }
        keys[i] = reinterpret_cast<uint32_t*>(w8 + lw.keys[i]);
    }
    const int sms = device_sm_count();
    if (sms <= 0) return cuda_fail(cudaGetLastError(), "querying the SM count");
    const cudaError_t e = launch_select_layers(sls.data(), keys.data(), n_layers,
                                               reinterpret_cast<int*>(w8 + lw.next_unit), sms, s);
    return e == cudaSuccess ? CKV_OK : cuda_fail(e, "launching the multi-layer selection kernel");
}

// ckv_score_windows(_lse): every layer's scores into io[i].scores, in one persistent launch.
ckv_status score_windows_impl(const ckv_config* cfg, int32_t n_layers, const ckv_layer_io* io,
                              const ckv_batch* batch, void* workspace, size_t workspace_bytes,
                              ckv_stream stream, bool given_lse) {
    static thread_local std::vector<Plan> pls;
    static thread_local std::vector<LayerJob> jobs;
    static thread_local std::vector<int64_t> tok, head;
    LayersWs lw;
    int T = 0;
    ckv_status st;
    if ((st = prepare_layers(cfg, n_layers, io, batch, pls, &T, &lw)) ||
        (st = check_layers_ws(lw, workspace, workspace_bytes, false)))
        return st;
    uint8_t* w8 = static_cast<uint8_t*>(workspace);
    if ((st = layer_jobs(pls, io, T, w8, lw, false, jobs, tok, head))) return st;
    if (given_lse && (st = layer_lse(pls, io, batch, jobs))) return st;
    return enqueue_layers(jobs, batch, T, w8 + lw.sums, reinterpret_cast<int*>(w8 + lw.counters),
                          reinterpret_cast<int*>(w8), -1, cfg->max_ctas,
                          reinterpret_cast<cudaStream_t>(stream));
}

}  // namespace

extern "C" {

ckv_status ckv_workspace_size_layers(const ckv_config* cfg, int32_t n_layers, const ckv_layer_io* io,
                                     const ckv_batch* batch, size_t* bytes) {
    std::vector<Plan> pls;
    LayersWs lw;
    int T = 0;
    ckv_status st = prepare_layers(cfg, n_layers, io, batch, pls, &T, &lw);
    if (st) return st;
    if (!bytes) return fail(CKV_ERR_INVALID_ARG, "bytes is NULL");
    *bytes = lw.total;
    return CKV_OK;
}

ckv_status ckv_score_windows(const ckv_config* cfg, int32_t n_layers, const ckv_layer_io* io,
                             const ckv_batch* batch, void* workspace, size_t workspace_bytes,
                             ckv_stream stream) {
    return score_windows_impl(cfg, n_layers, io, batch, workspace, workspace_bytes, stream, false);
}

ckv_status ckv_score_windows_lse(const ckv_config* cfg, int32_t n_layers, const ckv_layer_io* io,
                                 const ckv_batch* batch, void* workspace, size_t workspace_bytes,
                                 ckv_stream stream) {
    return score_windows_impl(cfg, n_layers, io, batch, workspace, workspace_bytes, stream, true);
}

ckv_status ckv_compress_layers(const ckv_config* cfg, int32_t n_layers, const ckv_layer_io* io,
                               const ckv_batch* batch, void* workspace, size_t workspace_bytes,
                               ckv_stream stream) {
    return compress_layers_impl(cfg, n_layers, io, batch, workspace, workspace_bytes, stream, false);
}

ckv_status ckv_compress_layers_lse(const ckv_config* cfg, int32_t n_layers, const ckv_layer_io* io,
                                   const ckv_batch* batch, void* workspace, size_t workspace_bytes,
                                   ckv_stream stream) {
    return compress_layers_impl(cfg, n_layers, io, batch, workspace, workspace_bytes, stream, true);
}

ckv_status ckv_semantic_retrieval_scores(const ckv_config* cfg, int32_t layer, const ckv_batch* batch,
                                         const void* q_dec, const void* k, int64_t tok_stride,
                                         int64_t head_stride, const float* lse, int64_t lse_head_stride,
                                         const uint8_t* in_answer, const int32_t* span, float* srs,
                                         void* workspace, size_t workspace_bytes, ckv_stream stream) {
    Plan pl;
    ckv_status st = make_plan(cfg, layer, pl);
    if (st) return st;
    int T = 0;
    WsLayout l;
    if ((st = check_batch(batch, &T)) || (st = resolve_strides(pl, &tok_stride, &head_stride)) ||
        (st = check_kv(q_dec, "q_dec", T)) || (st = check_kv(k, "k", T)) ||
        (st = check_ws(pl, batch, T, workspace, workspace_bytes, &l)) ||
        (st = check_lse(pl, batch, lse, &lse_head_stride)))
        return st;
    if (!in_answer || !span || !srs) return fail(CKV_ERR_INVALID_ARG, "in_answer, span and srs are required");
    if (!aligned(span, 4) || !aligned(srs, 4)) return fail(CKV_ERR_INVALID_ARG, "span or srs is misaligned");
    cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
    uint8_t* w8 = static_cast<uint8_t*>(workspace);
    SrsLaunch L;
    memset(&L, 0, sizeof L);
    L.lse = lse;
    L.lse_stride = lse_head_stride;
    L.in_answer = in_answer;
    float* scores = reinterpret_cast<float*>(w8 + l.scores);
    L.lse_masked = reinterpret_cast<float*>(w8 + l.srs_lse);
    L.scores = scores;
    L.span = span;
    L.cu_seqlens_dev = batch->cu_seqlens_dev;
    L.sel_heads = pl.sel_heads.data();
    L.srs = srs;
    L.status = static_cast<int*>(workspace);
    L.S = batch->num_seqs;
    L.T = T;
    L.Hq = pl.Hq;
    L.w = pl.w;
    L.n_sel = pl.n_sel;
    cudaError_t e = launch_srs_mask(L, s);
    if (e != cudaSuccess) return cuda_fail(e, "launching the lse mask kernel");
    if ((st = enqueue_score(pl, batch, T, q_dec, k, tok_stride, head_stride, scores, workspace, l, -1, s,
                            kMaxScoreItems, L.lse_masked, static_cast<int64_t>(batch->num_seqs) * pl.w)))
        return st;
    e = launch_srs_span(L, s);
    return e == cudaSuccess ? CKV_OK : cuda_fail(e, "launching the span-sum kernel");
}

ckv_status ckv_read_device_status(void* workspace, ckv_stream stream, int32_t reset,
                                  int32_t* code, int32_t* detail) {
    if (!workspace || !code) return fail(CKV_ERR_INVALID_ARG, "workspace and code are required");
    cudaError_t e = cudaStreamSynchronize(reinterpret_cast<cudaStream_t>(stream));
    if (e != cudaSuccess) return cuda_fail(e, "synchronising the stream");
    int32_t hdr[2] = {0, 0};
    e = cudaMemcpy(hdr, workspace, sizeof hdr, cudaMemcpyDeviceToHost);
    if (e != cudaSuccess) return cuda_fail(e, "reading the status word");
    *code = hdr[0];
    if (detail) *detail = hdr[1];
    if (reset) {
        e = cudaMemset(workspace, 0, sizeof hdr);
        if (e != cudaSuccess) return cuda_fail(e, "clearing the status word");
    }
    return CKV_OK;
}

// ---------------------------------------------------------------------- no-allocation variant
// The scratch of ckv_score_window_static: a status header followed by the per-chunk softmax
// partials (float2 per window-row column, kMaxCols columns per work item).
static __device__ __align__(256) unsigned char g_score_scratch[CKV_STATIC_SCRATCH_BYTES];

namespace {
constexpr int kMaxDevices = 64;
std::once_flag g_scratch_once[kMaxDevices];
void* g_scratch_addr[kMaxDevices] = {};
cudaError_t g_scratch_err[kMaxDevices] = {};
}  // namespace

ckv_status ckv_score_window_static(const ckv_config* cfg, int32_t layer, const ckv_batch* batch,
                                   const void* q_win, const void* k, int64_t tok_stride,
                                   int64_t head_stride, float* scores, int32_t* status_out,
                                   ckv_stream stream) {
    static_assert(sizeof(WsHeader) == 256, "header");
    Plan pl;
    ckv_status st = make_plan(cfg, layer, pl);
    if (st) return st;
    int T = 0;
    if ((st = check_batch(batch, &T)) || (st = resolve_strides(pl, &tok_stride, &head_stride)) ||
        (st = check_kv(q_win, "q_win", T)) || (st = check_kv(k, "k", T)) ||
        (st = check_kv(scores, "scores", T)))
        return st;
    if (status_out && !aligned(status_out, 4))
        return fail(CKV_ERR_INVALID_ARG, "status_out is not 4-byte aligned");
    int dev = -1;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return cuda_fail(e, "cudaGetDevice");
    if (dev < 0 || dev >= kMaxDevices) return fail(CKV_ERR_UNSUPPORTED, "device index %d", dev);
    int ctas = device_sm_count();
    if (ctas <= 0) return cuda_fail(cudaGetLastError(), "querying the SM count");
    if (pl.max_ctas > 0) ctas = std::min(ctas, pl.max_ctas);  // the CTAs enqueue_score plans for
    bool resident = false;
    if ((st = resident_choice(pl, batch, -1, std::min(ctas, CKV_STATIC_SCRATCH_ITEMS), &resident)))
        return st;
    if (resident) {
        // The same plan as the launch below makes: its work items, over all of its launches,
        // must fit the array (each launch's items are also bounded by the array's size).
        static thread_local ScoreLaunch probe;
        if ((st = plan_score(pl, batch, -1, std::min(ctas, CKV_STATIC_SCRATCH_ITEMS), probe,
                             CKV_STATIC_SCRATCH_ITEMS)))
            return st;
        const int n_items = static_cast<int>(probe.items.size());
        if (n_items > CKV_STATIC_SCRATCH_ITEMS)
            return fail(CKV_ERR_UNSUPPORTED,
                        "this batch needs %d scratch work items; the static scratch holds %d "
                        "(use ckv_score_window with a workspace)", n_items, CKV_STATIC_SCRATCH_ITEMS);
    } else {
        // The two-pass kernel's exchange: one fp64 sum per column and a counter per (head
        // batch, sequence) unit of a launch (a launch takes launch_seq_chunk sequences).
        const int units = pl.nb * std::min(batch->num_seqs, launch_seq_chunk(pl.nb));
        if (units > CKV_STATIC_SCRATCH_UNITS)
            return fail(CKV_ERR_UNSUPPORTED,
                        "this batch needs %d scratch units; the static scratch holds %d "
                        "(use ckv_score_window with a workspace)", units, CKV_STATIC_SCRATCH_UNITS);
    }
    // Once per device, with that device current: the device address of the scratch array.
    std::call_once(g_scratch_once[dev], [dev] {
        void* ptr = nullptr;
        g_scratch_err[dev] = cudaGetSymbolAddress(&ptr, g_score_scratch);
        g_scratch_addr[dev] = ptr;
    });
    if (g_scratch_err[dev] != cudaSuccess || !g_scratch_addr[dev])
        return cuda_fail(g_scratch_err[dev], "cudaGetSymbolAddress of the static scratch");
    void* scratch = g_scratch_addr[dev];
    cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
    e = cudaMemsetAsync(scratch, 0, 2 * sizeof(int32_t), s);  // the status word starts at zero
    if (e != cudaSuccess) return cuda_fail(e, "clearing the static status word");
    // Layout: the status header, then either kernel's exchange (they never run in one call).
    static_assert(CKV_STATIC_SCRATCH_ITEMS * kMaxCols * sizeof(float2) ==
                      CKV_STATIC_SCRATCH_UNITS * kMaxCols * sizeof(double), "scratch regions");
    WsLayout l;
    l.header = 0;
    l.partials = sizeof(WsHeader);
    l.counters = l.partials + static_cast<size_t>(CKV_STATIC_SCRATCH_ITEMS) * kMaxCols * sizeof(float2);
    l.sums = l.partials;
    l.unit_counters = l.counters;
    l.total = CKV_STATIC_SCRATCH_BYTES;
    if ((st = enqueue_score(pl, batch, T, q_win, k, tok_stride, head_stride, scores, scratch, l, -1, s,
                            CKV_STATIC_SCRATCH_ITEMS)))
        return st;
    if (status_out) {
        e = cudaMemcpyAsync(status_out, scratch, 2 * sizeof(int32_t), cudaMemcpyDeviceToDevice, s);
        if (e != cudaSuccess) return cuda_fail(e, "copying the static status word");
    }
    return CKV_OK;
}

}  // extern "C"
