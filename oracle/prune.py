"""Performance-aware expert pruning scores (arXiv 2509.25689 Sec. 3.1) —
TEST INFRASTRUCTURE ONLY.

Plain-Python statement of the expert-importance score, for checking the
library's host routine.  Only ``tests/`` may import it.

Over a calibration stream of n_tokens routed tokens (expert ids idx[t, j]
and routing weights w[t, j], j < top_k):
  f_e  = (number of tokens that select e) / n_tokens   (activation frequency)
  s_e  = mean of w[t, j] over the selections of e, 0 if e is never selected
         (average routing score assigned to e when selected)
  I_e  = alpha * f_e + (1 - alpha) * s_e
and the ceil(r E) experts of largest I_e are kept (ties to the lower id),
returned in ascending id order.
Readings: the score is the weight the router assigns to the slot (the
normalised, scaled combine weight).  The paper fixes no summation order, so
the sum of e's weights is taken order-free: every weight is rounded to the
nearest multiple of 2^-64 (ties to even; exact for |w| >= 2^-40, which
covers every routing weight in practice), the multiples are added exactly
as integers, and the total is rounded once to double; s_e is that double
divided by the count (one IEEE division) and f_e the count over n_tokens.
Any accumulation order, on any device, then gives the same bits.
ceil(r E) is taken with the same 1e-12 guard as the activation adjustment.
"""
from __future__ import annotations

import math


FIX_BITS = 64          # fractional bits of the weight accumulator


def fixed_weight(w):
    """w rounded to the nearest multiple of 2^-64 (ties to even), as an
    integer count of 2^-64 units.  float * 2^64 is exact (a power of two);
    round() on a float rounds half to even."""
    return round(float(w) * 2.0 ** FIX_BITS)


def expert_counts_and_sums(idx, w, n_experts):
    """Integer selection counts and exact fixed-point weight sums per expert."""
    count = [0] * n_experts
    fsum = [0] * n_experts
    for t in range(len(idx)):
        for j in range(len(idx[t])):
            e = int(idx[t][j])
            count[e] += 1
            fsum[e] += fixed_weight(w[t][j])
    return count, fsum


def expert_importance(idx, w, n_experts, alpha):
    """idx, w: sequences of rows (one per token) of top_k entries."""
    n_tokens = len(idx)
    count, fsum = expert_counts_and_sums(idx, w, n_experts)
    scores = []
    for e in range(n_experts):
        f = count[e] / n_tokens if n_tokens > 0 else 0.0
        # int / int is correctly rounded in Python: the exact sum, rounded once
        s = (fsum[e] / 2 ** FIX_BITS) / count[e] if count[e] > 0 else 0.0
        scores.append(alpha * f + (1.0 - alpha) * s)
    return scores


def keep_count(r, n_experts):
    return int(math.ceil(r * n_experts - 1e-12))


def prune(idx, w, n_experts, alpha, r):
    scores = expert_importance(idx, w, n_experts, alpha)
    k = keep_count(r, n_experts)
    order = sorted(range(n_experts), key=lambda e: (-scores[e], e))
    return sorted(order[:k]), scores
