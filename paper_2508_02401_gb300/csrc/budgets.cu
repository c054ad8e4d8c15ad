// Layer budgets of the paper's error-aware, layer-adaptive allocation (arxiv 2508.02401,
// App. B): the per-layer error scores of Eq. 11-13 and Algorithm 1.  Host code only.
#include "ckv.h"

#include <math.h>

#include <algorithm>
#include <numeric>
#include <vector>

namespace ckv {
ckv_status set_error(ckv_status st, const char* fmt, ...);
}

extern "C" {

CKV_API ckv_status ckv_layer_error_scores(const double* errors, int32_t num_datasets,
                                          int32_t num_layers, double* scores) {
    if (!errors || !scores) return ckv::set_error(CKV_ERR_INVALID_ARG, "errors and scores are required");
    if (num_datasets < 1 || num_layers < 1)
        return ckv::set_error(CKV_ERR_INVALID_ARG, "need at least one dataset and one layer");
    std::vector<double> mean(num_layers, 0.0);
    for (int32_t d = 0; d < num_datasets; ++d) {
        const double* row = errors + static_cast<size_t>(d) * num_layers;
        double total = 0.0;
        for (int32_t l = 0; l < num_layers; ++l) {
            if (!isfinite(row[l]) || row[l] < 0.0)
                return ckv::set_error(CKV_ERR_INVALID_ARG, "error %d,%d is negative or not finite", d, l);
            total += row[l];
        }
        if (total == 0.0) return ckv::set_error(CKV_ERR_INVALID_ARG, "the errors of dataset %d sum to 0", d);
        for (int32_t l = 0; l < num_layers; ++l) mean[l] += row[l] / total;  // Eq. 11, summed for Eq. 12
    }
    double total = 0.0;
    for (int32_t l = 0; l < num_layers; ++l) {
        mean[l] /= num_datasets;  // Eq. 12
        total += mean[l];
    }
    if (total == 0.0) return ckv::set_error(CKV_ERR_INVALID_ARG, "the scores sum to 0");
    for (int32_t l = 0; l < num_layers; ++l) scores[l] = mean[l] / total;  // Eq. 13
    return CKV_OK;
}

CKV_API ckv_status ckv_allocate_budgets(const double* scores, int32_t num_layers,
                                        int64_t total_budget, int32_t min_budget,
                                        int32_t max_budget, int32_t* budgets) {
    if (!scores || !budgets) return ckv::set_error(CKV_ERR_INVALID_ARG, "scores and budgets are required");
    if (num_layers < 1) return ckv::set_error(CKV_ERR_INVALID_ARG, "num_layers %d < 1", num_layers);
    if (min_budget < 0 || max_budget < min_budget)
        return ckv::set_error(CKV_ERR_INVALID_ARG, "need 0 <= min_budget <= max_budget");
    for (int32_t l = 0; l < num_layers; ++l)
        if (!isfinite(scores[l]) || scores[l] < 0.0)
            return ckv::set_error(CKV_ERR_INVALID_ARG, "score %d is negative or not finite", l);
    const int64_t m = min_budget, M = max_budget;
    // every layer at m, the rest in proportion to the scores, rounded (ties to even) and clipped
    const int64_t R = total_budget - m * num_layers;
    std::vector<int64_t> B(num_layers);
    int64_t sum = 0;
    for (int32_t l = 0; l < num_layers; ++l) {
        const double share = nearbyint(scores[l] * static_cast<double>(R));
        B[l] = std::min(std::max(m + static_cast<int64_t>(share), m), M);
        sum += B[l];
    }
    // Settle the difference one token at a time: the loop of Algorithm 1 keeps choosing the
    // same layer (highest score below M, or lowest score above m; lowest index on ties) until
    // it reaches its bound, so it fills the layers in that order.
    int64_t delta = total_budget - sum;
    if (delta != 0) {
        std::vector<int32_t> order(num_layers);
        std::iota(order.begin(), order.end(), 0);
        if (delta > 0)
            std::stable_sort(order.begin(), order.end(),
                             [&](int32_t a, int32_t b) { return scores[a] > scores[b]; });
        else
            std::stable_sort(order.begin(), order.end(),
                             [&](int32_t a, int32_t b) { return scores[a] < scores[b]; });
        for (int32_t i : order) {
            if (delta == 0) break;
            if (delta > 0) {
                const int64_t add = std::min(delta, M - B[i]);
                B[i] += add;
                delta -= add;
            } else {
                const int64_t sub = std::min(-delta, B[i] - m);
                B[i] -= sub;
                delta += sub;
            }
        }
    }
    for (int32_t l = 0; l < num_layers; ++l) budgets[l] = static_cast<int32_t>(B[l]);
    return CKV_OK;
}

}  // extern "C"
