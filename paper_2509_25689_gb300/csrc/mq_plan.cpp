// Tensor-level mixed-precision planner (arXiv 2509.25689 Sec. 3.3): budget,
// size-class upgrades in sensitivity order and the three-stage back-off.
// Host code; the rules and the exact integer cost model are stated in
// include/moeq_plan.h.
#include <algorithm>
#include <cmath>
#include <cstdint>
#include <queue>
#include <vector>

#include "moeq.h"
#include "moeq_plan.h"

namespace {

// Breadth-first bisection of [0, n): the midpoint of each interval's
// boundaries, rounded up, then its two halves.
void bp_order(int32_t n, std::vector<int32_t>& out) {
    out.clear();
    out.reserve(n > 0 ? n : 0);
    std::vector<std::pair<int32_t, int32_t>> q;
    q.reserve(n > 0 ? 2 * n + 1 : 1);
    q.emplace_back(0, n);
    for (size_t h = 0; h < q.size(); ++h) {
        const int32_t lo = q[h].first, hi = q[h].second;
        if (hi <= lo) continue;
        const int32_t mid = std::min<int32_t>(lo + (hi - lo + 1) / 2, hi - 1);
        out.push_back(mid);
        q.emplace_back(lo, mid);
        q.emplace_back(mid + 1, hi);
    }
}

}  // namespace

extern "C" int mq_binary_partition_order(int32_t n, int32_t* order_out) {
    if (n < 0 || (n > 0 && order_out == nullptr)) return MQ_EINVAL;
    std::vector<int32_t> o;
    bp_order(n, o);
    std::copy(o.begin(), o.end(), order_out);
    return MQ_OK;
}

extern "C" int mq_plan_precision(const mq_plan_cfg* cfg, const mq_plan_tensor* tensors, int32_t n,
                                 int32_t* level_out, int64_t* total_bits64_out) {
    if (cfg == nullptr || n < 0 || (n > 0 && (tensors == nullptr || level_out == nullptr))) return MQ_EINVAL;
    const int32_t L = cfg->n_levels;
    if (L < 1 || L > 64 || cfg->bits64 == nullptr || cfg->mem_limit_bytes < 0) return MQ_EINVAL;
    const int32_t* b = cfg->bits64;
    for (int32_t l = 0; l < L; ++l)
        if (b[l] <= 0 || b[l] > 4096 || (l > 0 && b[l] <= b[l - 1])) return MQ_EINVAL;
    auto in = [&](int32_t v) { return v >= 0 && v < L; };
    if (!in(cfg->low) || !in(cfg->lowest) || cfg->lowest > cfg->low || !in(cfg->small_level) ||
        !in(cfg->medium_level) || !in(cfg->floor_level))
        return MQ_EINVAL;
    // at most 2^48 parameters in all and 64 bits per weight: totals stay below 2^60
    int64_t all_params = 0;
    for (int32_t i = 0; i < n; ++i) {
        const mq_plan_tensor& t = tensors[i];
        if (t.params < 0 || t.kind < 0 || t.kind > 3 || !std::isfinite(t.sens)) return MQ_EINVAL;
        if (t.params > (int64_t(1) << 48) - all_params) return MQ_EINVAL;
        all_params += t.params;
    }
    const int32_t floor_l = std::max(cfg->floor_level, cfg->low + 1);   // upgraded tensors stay above Q_low
    const int64_t limit = cfg->mem_limit_bytes > INT64_MAX / 512 ? INT64_MAX : 512 * cfg->mem_limit_bytes;

    std::vector<int32_t> level(n, cfg->low);
    int64_t total = 0;
    for (int32_t i = 0; i < n; ++i) total += tensors[i].params * b[cfg->low];
    auto set_level = [&](int32_t i, int32_t l) {
        total += tensors[i].params * (int64_t(b[l]) - b[level[i]]);
        level[i] = l;
    };
    auto fits = [&]() { return total <= limit; };

    // routed back-off steps: gate & up of each routed layer in binary-partition
    // order, then the down tensors in the same order
    std::vector<int32_t> layers;
    for (int32_t i = 0; i < n; ++i)
        if (tensors[i].kind != MQ_TENSOR_OTHER) layers.push_back(tensors[i].layer);
    std::sort(layers.begin(), layers.end());
    layers.erase(std::unique(layers.begin(), layers.end()), layers.end());
    std::vector<int32_t> pos;
    bp_order((int32_t)layers.size(), pos);
    std::vector<int32_t> rank_of_layer_pos(layers.size());
    for (size_t r = 0; r < pos.size(); ++r) rank_of_layer_pos[pos[r]] = (int32_t)r;
    // step index of each routed tensor; steps [0, nl) gate/up, [nl, 2 nl) down
    const int32_t nl = (int32_t)layers.size();
    std::vector<std::vector<int32_t>> steps(2 * (size_t)nl);
    for (int32_t i = 0; i < n; ++i) {
        const mq_plan_tensor& t = tensors[i];
        if (t.kind == MQ_TENSOR_OTHER) continue;
        const int32_t p = (int32_t)(std::lower_bound(layers.begin(), layers.end(), t.layer) - layers.begin());
        const int32_t r = rank_of_layer_pos[p];
        steps[(t.kind == MQ_TENSOR_EXPERT_DOWN ? nl : 0) + r].push_back(i);
    }
    size_t next_step = 0;
    while (next_step < steps.size() && steps[next_step].empty()) ++next_step;

    auto target = [&](int32_t i) -> int32_t {
        const int64_t p = tensors[i].params;
        if (p < cfg->small_max) return cfg->small_level;
        if (p <= cfg->medium_max) return cfg->medium_level;
        return cfg->low;
    };
    std::vector<int32_t> cands;
    for (int32_t i = 0; i < n; ++i)
        if (tensors[i].kind == MQ_TENSOR_OTHER && target(i) > cfg->low) cands.push_back(i);
    std::stable_sort(cands.begin(), cands.end(),
                     [&](int32_t a, int32_t c) { return tensors[a].sens > tensors[c].sens; });

    // earlier upgrades above the floor, largest first (ties: upgraded earlier)
    using Key = std::pair<int64_t, int64_t>;   // (params, -upgrade order)
    std::priority_queue<std::pair<Key, int32_t>> big;
    int64_t n_up = 0;
    for (const int32_t i : cands) {
        set_level(i, target(i));
        if (!fits()) {   // (1) local: one level down, then a second
            for (int k = 0; k < 2; ++k) {
                const int32_t l = level[i] - 1;
                if (l >= floor_l) set_level(i, l);
                if (fits()) break;
            }
        }
        while (!fits() && !big.empty()) {   // (2) global: the largest earlier upgrade
            const int32_t j = big.top().second;
            if (level[j] <= floor_l) { big.pop(); continue; }
            set_level(j, level[j] - 1);
        }
        while (!fits() && next_step < steps.size()) {   // (3) routed experts to Q_low'
            for (const int32_t j : steps[next_step]) set_level(j, cfg->lowest);
            ++next_step;
            while (next_step < steps.size() && steps[next_step].empty()) ++next_step;
        }
        if (!fits()) {
            set_level(i, cfg->low);
            continue;
        }
        big.push({{tensors[i].params, -n_up}, i});
        ++n_up;
    }
    std::copy(level.begin(), level.end(), level_out);
    if (total_bits64_out) *total_bits64_out = total;
    return MQ_OK;
}

// Activation adjustment (Sec. 3.2): k_pruned = ceil(r k_orig) per layer, then
// one expert at a time off the layers in binary-partition order (cycling,
// none below 1) until 2 sum k_i P_i fits the budget.
extern "C" int mq_activation_plan(int32_t k_orig, double retain, int32_t n_layers, const int64_t* params_per_expert,
                                  int64_t flops_budget, int32_t* k_out, int64_t* flops_out) {
    if (k_orig < 1 || k_orig > 256 || !(retain > 0.0 && retain <= 1.0) || n_layers < 0 || n_layers > 4096 ||
        flops_budget < 0)
        return MQ_EINVAL;
    if (n_layers > 0 && (params_per_expert == nullptr || k_out == nullptr)) return MQ_EINVAL;
    for (int32_t i = 0; i < n_layers; ++i)
        if (params_per_expert[i] < 1 || params_per_expert[i] > (int64_t(1) << 40)) return MQ_EINVAL;
    const int32_t kp = (int32_t)std::ceil(retain * k_orig - 1e-12);
    std::vector<int32_t> k(n_layers, kp);
    // 2 * 256 * 2^40 * 4096 < 2^63
    int64_t flops = 0;
    for (int32_t i = 0; i < n_layers; ++i) flops += 2 * (int64_t)kp * params_per_expert[i];
    std::vector<int32_t> order;
    bp_order(n_layers, order);
    int64_t above_one = kp > 1 ? n_layers : 0;   // layers that can still give up an expert
    for (size_t pos = 0; flops > flops_budget && above_one > 0; ++pos) {
        const int32_t l = order[pos % order.size()];
        if (k[l] > 1) {
            --k[l];
            flops -= 2 * params_per_expert[l];
            if (k[l] == 1) --above_one;
        }
    }
    std::copy(k.begin(), k.end(), k_out);
    if (flops_out) *flops_out = flops;
    return MQ_OK;
}
