// Expert-importance scores for performance-aware expert pruning (arXiv
// 2509.25689 Sec. 3.1): I_e = alpha f_e + (1 - alpha) s_e over a routed
// calibration stream, and the ceil(r E) experts kept.  Host code; the
// definitions are stated in include/moeq_plan.h.
#include <algorithm>
#include <cmath>
#include <cstdint>
#include <numeric>
#include <vector>

#include "moeq.h"
#include "moeq_plan.h"
#include "mq_fixsum.h"

extern "C" int mq_expert_importance(const int32_t* topk_idx, const float* topk_w, int32_t n_tokens, int32_t top_k,
                                    int32_t n_experts, double alpha, double retain, double* scores_out,
                                    int32_t* keep_out, int32_t* n_keep_out) {
    if (n_tokens < 0 || top_k < 1 || n_experts < 1 || n_experts > (1 << 20)) return MQ_EINVAL;
    if (!(alpha >= 0.0 && alpha <= 1.0) || !(retain > 0.0 && retain <= 1.0)) return MQ_EINVAL;
    if (n_tokens > 0 && (topk_idx == nullptr || topk_w == nullptr)) return MQ_EINVAL;
    if (keep_out == nullptr || n_keep_out == nullptr) return MQ_EINVAL;
    const size_t n = (size_t)n_tokens * (size_t)top_k;
    std::vector<mq::Fix128> wfix(n);
    for (size_t i = 0; i < n; ++i)
        if (topk_idx[i] < 0 || topk_idx[i] >= n_experts || !mq::fix_from_float(topk_w[i], wfix[i])) return MQ_EINVAL;

    // counts, and weight sums exact in 2^-64 units (order-free)
    std::vector<int64_t> count(n_experts, 0);
    std::vector<mq::Fix128> ssum(n_experts, mq::Fix128{0, 0});
    for (size_t i = 0; i < n; ++i) {
        count[topk_idx[i]] += 1;
        mq::fix_add(ssum[topk_idx[i]], wfix[i]);
    }
    std::vector<double> score(n_experts);
    for (int32_t e = 0; e < n_experts; ++e) {
        const double f = n_tokens > 0 ? (double)count[e] / (double)n_tokens : 0.0;
        const double s = count[e] > 0 ? mq::fix_to_double(ssum[e]) / (double)count[e] : 0.0;
        score[e] = alpha * f + (1.0 - alpha) * s;
    }
    const int32_t k = (int32_t)std::ceil(retain * n_experts - 1e-12);
    std::vector<int32_t> order(n_experts);
    std::iota(order.begin(), order.end(), 0);
    std::stable_sort(order.begin(), order.end(), [&](int32_t a, int32_t b) { return score[a] > score[b]; });
    order.resize(k);
    std::sort(order.begin(), order.end());
    std::copy(order.begin(), order.end(), keep_out);
    *n_keep_out = k;
    if (scores_out) std::copy(score.begin(), score.end(), scores_out);
    return MQ_OK;
}
