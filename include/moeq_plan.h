/*
 * moeq_plan — host-side compression planning, C ABI: the tensor-level
 * mixed-precision planner and the expert-importance scores for pruning.
 *
 * Chooses a quantization level for every tensor of a model under a memory
 * limit, following arXiv 2509.25689 Sec. 3.3 ("Hardware-Constrained Budget
 * Formulation", "Dynamic Allocation with Back-off"):
 *   - every tensor starts at the base level Q_low; the model then costs
 *     S_low, and the upgrade budget is B_base = M_limit - S_low plus what
 *     routed-expert downgrades to Q_low' free (B_delta);
 *   - tensors that are not routed-expert tensors are taken in descending
 *     sensitivity Sens(t) and raised to a level set by their size: fewer
 *     than small_max parameters -> small_level (Q8), up to medium_max ->
 *     medium_level (Q6), larger ones stay at Q_low; routed-expert tensors
 *     are never raised;
 *   - when an upgrade breaks the budget: (1) the tensor goes down one level,
 *     then a second; (2) the largest earlier-upgraded tensor goes down one
 *     level, repeatedly, none below floor_level (Q4: a Q8 tensor goes down
 *     at most three levels); (3) routed-expert tensors go from Q_low to
 *     Q_low', gate and up of one layer per step in binary-partition layer
 *     order, then the down tensors in the same order; if the budget still
 *     fails the tensor stays at Q_low.
 * Costs are exact integers: a level's width is given in 1/64 bit per weight
 * (every k-quant width is a multiple of 1/64), and a plan fits when
 * sum |t| * bits64[level_t] <= 512 * mem_limit_bytes.
 *
 * No back-off step takes an upgraded tensor down to Q_low or below.
 *
 * Conventions: host pointers, caller-owned buffers; returns MQ_OK (0) or
 * MQ_EINVAL (-1) for a null pointer, a negative size, a level index out of
 * range, widths not strictly ascending in 1..4096, more than 2^48
 * parameters in all, a non-finite sensitivity or a tensor kind other than
 * 0..3; nothing is written on error.  No GPU is used.
 */
#ifndef MOEQ_PLAN_H
#define MOEQ_PLAN_H

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

enum { MQ_TENSOR_OTHER = 0, MQ_TENSOR_EXPERT_GATE = 1, MQ_TENSOR_EXPERT_UP = 2, MQ_TENSOR_EXPERT_DOWN = 3 };

/* One tensor: parameter count |t|, its layer, its kind (MQ_TENSOR_*; the
 * routed-expert kinds stand for the routed experts' tensors of that layer)
 * and its sensitivity Sens(t) (any finite value; larger = upgraded first). */
typedef struct {
    int64_t params;
    int32_t layer;
    int32_t kind;
    double sens;
} mq_plan_tensor;

/* The level ladder and the rules.  bits64[0..n_levels-1]: width of each
 * level in 1/64 bit per weight, strictly ascending (e.g. IQ1_S 100, IQ1_M
 * 112, Q2_K 168, Q3_K 220, Q4_K 288, Q5_K 352, Q6_K 420, Q8_0 544).
 * lowest <= low < n_levels; small_level, medium_level, floor_level <
 * n_levels.  mem_limit_bytes: M_limit in bytes (>= 0). */
typedef struct {
    int32_t n_levels;
    const int32_t* bits64;
    int32_t low, lowest, small_level, medium_level, floor_level;
    int64_t small_max, medium_max;
    int64_t mem_limit_bytes;
} mq_plan_cfg;

/* Plans n tensors.  level_out: host int32 [n], the chosen level index of
 * every tensor; total_bits64_out (or NULL): sum |t| * bits64[level_t] of the
 * plan (the plan fits when this is <= 512 * mem_limit_bytes). */
int mq_plan_precision(const mq_plan_cfg* cfg, const mq_plan_tensor* tensors, int32_t n, int32_t* level_out,
                      int64_t* total_bits64_out);

/* Binary-partition order of n layer positions (Sec. 3.3 back-off rule 3):
 * the position at the midpoint of [lo, hi) rounded up (clamped to hi - 1),
 * then the halves [lo, mid) and [mid + 1, hi), breadth first; for n = 58
 * it starts 29, 15, 44, 8.  order_out: host int32 [n], a permutation of
 * 0..n-1.  n >= 0. */
int mq_binary_partition_order(int32_t n, int32_t* order_out);

/* Hardware-aware activation adjustment (Sec. 3.2).  After pruning to a
 * retention ratio retain, every layer activates k_pruned = ceil(retain *
 * k_orig - 1e-12) experts per token; per device the per-layer counts
 * k_i <= k_pruned are tuned so that FLOPs_active = 2 sum_i k_i P_i (P_i =
 * params_per_expert[i], one expert of layer i) fits flops_budget: starting
 * from k_pruned everywhere, one layer at a time gives up one expert, the
 * layers taken in binary-partition order (as mq_binary_partition_order,
 * cycling through it), none below 1.  k_out: host int32 [n_layers];
 * flops_out (or NULL): FLOPs_active of the plan, above flops_budget only when
 * every k_i is 1.  k_orig in 1..256, retain in (0, 1], n_layers in 0..4096,
 * every P_i in 1..2^40, flops_budget >= 0; MQ_OK or MQ_EINVAL (nothing
 * written).  topk_group needs no change: k_i never rises. */
int mq_activation_plan(int32_t k_orig, double retain, int32_t n_layers, const int64_t* params_per_expert,
                       int64_t flops_budget, int32_t* k_out, int64_t* flops_out);

/* Expert-importance scores for pruning (Sec. 3.1).  Over a routed
 * calibration stream of n_tokens tokens (moe_quant_route's topk_idx /
 * topk_w copied to the host: int32 / fp32 [n_tokens, top_k], ids in
 * 0..n_experts-1, finite weights with |w| < 2^32):
 *   f_e = tokens selecting e / n_tokens, s_e = mean weight of e's
 *   selections (0 if none), I_e = alpha f_e + (1 - alpha) s_e.
 * The weight sum of e is order-free: every weight rounded to the nearest
 * multiple of 2^-64 (ties to even; exact for |w| >= 2^-40), the multiples
 * added exactly, the total rounded once to double and divided by the count.
 * The device histogram (moeq_stats.h) gives the same bits.
 * The ceil(retain * n_experts) experts of largest I_e (ties to the lower id)
 * are kept: keep_out (host int32, room for n_experts) receives their ids in
 * ascending order and *n_keep_out their number; scores_out (host double
 * [n_experts], or NULL) receives I_e.  alpha in [0, 1], retain in (0, 1].
 * Returns MQ_OK or MQ_EINVAL (nothing written). */
int mq_expert_importance(const int32_t* topk_idx, const float* topk_w, int32_t n_tokens, int32_t top_k,
                         int32_t n_experts, double alpha, double retain, double* scores_out, int32_t* keep_out,
                         int32_t* n_keep_out);

#ifdef __cplusplus
}
#endif
#endif
