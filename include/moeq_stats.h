/*
 * moeq_stats — device histogram of routed experts for performance-aware
 * expert pruning (arXiv 2509.25689 Sec. 3.1), C ABI.
 *
 * Sec. 3.1 scores every routed expert of the unpruned model over a
 * calibration stream: its activation frequency f_e (the share of tokens
 * that select it), its average routing score s_e (the mean routing weight
 * of its selections) and the importance I_e = alpha f_e + (1 - alpha) s_e;
 * the ceil(r E) experts of largest I_e are kept (r = 0.75 in Sec. 4.1).
 * Here the counts and weight sums are accumulated on the GPU from the
 * router's device outputs (moe_quant_route's or moe_quant_forward's
 * topk_idx / topk_w), batch after batch, without copying them to the host.
 *
 * Accumulation is deterministic and order-free: counts are integers, and
 * every weight is rounded to the nearest multiple of 2^-64 (ties to even;
 * exact for any float32 with |w| >= 2^-40) and added as a 128-bit integer.
 * The scores are therefore bit-identical to mq_expert_importance
 * (moeq_plan.h) on the same stream, however it is split into batches.
 *
 * Statistics buffer (device memory, 16-byte aligned, caller-owned,
 * mq_expert_stats_bytes(n_experts) bytes):
 *   offset 0            uint64 n_tokens       tokens added so far
 *   offset 8            uint32 err_bits       1: an expert id outside
 *                                             0..n_experts-1 was skipped;
 *                                             2: a weight that is not finite
 *                                             or has |w| >= 2^32 was skipped
 *   offset 12           uint32 (reserved, 0)
 *   offset 16           uint64 count[n_experts]    selections of expert e
 *   then                uint64 wsum_lo[n_experts]  weight sum of e in units of
 *   then                int64  wsum_hi[n_experts]  2^-64: wsum_hi * 2^64 + wsum_lo
 *                                                  (two's complement)
 * Conventions: device pointers except where stated; every call enqueues on
 * cuda_stream (NULL = legacy default stream) and returns without waiting.
 * Returns MQ_OK, MQ_EINVAL (null pointer, n_experts outside 1..1024,
 * n_tokens < 0, top_k outside 1..32, alpha outside [0, 1], retain outside
 * (0, 1]; nothing enqueued), MQ_EALIGN (a buffer not 16-byte aligned; for
 * topk_idx / topk_w 4 bytes suffice) or MQ_ECUDA (a launch failed).
 */
#ifndef MOEQ_STATS_H
#define MOEQ_STATS_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* Bytes of a statistics buffer for n_experts experts (16 + 24 n_experts;
 * 0 for n_experts outside 1..1024). */
size_t mq_expert_stats_bytes(int32_t n_experts);

/* Clears the buffer (all counts, sums, the token count and err_bits). */
int mq_expert_stats_reset(void* stats, int32_t n_experts, void* cuda_stream);

/* Adds one routed batch: topk_idx int32 / topk_w fp32 [n_tokens, top_k]
 * row-major.  n_tokens = 0 enqueues nothing. */
int mq_expert_stats_add(void* stats, int32_t n_experts, const int32_t* topk_idx, const float* topk_w,
                        int32_t n_tokens, int32_t top_k, void* cuda_stream);

/* Scores from the statistics so far:
 *   freq   double [n_experts] or NULL: f_e = count_e / n_tokens (0 when no
 *          token was added);
 *   mean_w double [n_experts] or NULL: s_e = (wsum_e rounded to double) /
 *          count_e, 0 when count_e = 0;
 *   scores double [n_experts] or NULL: I_e = alpha f_e + (1 - alpha) s_e,
 *          each product and the sum rounded separately (no fused multiply-add);
 *   keep   int32 [ceil(retain n_experts)] or NULL: the ids of the
 *          ceil(retain n_experts) largest I_e (ties to the lower id), in
 *          ascending order;
 *   n_keep host int32* or NULL: receives ceil(retain n_experts) (computed on
 *          the host as ceil(retain * n_experts - 1e-12)).
 * One CTA; reads the buffer after the work enqueued before it. */
int mq_expert_stats_scores(const void* stats, int32_t n_experts, double alpha, double retain, double* freq,
                           double* mean_w, double* scores, int32_t* keep, int32_t* n_keep, void* cuda_stream);

#ifdef __cplusplus
}
#endif
#endif
