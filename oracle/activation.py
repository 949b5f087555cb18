"""Hardware-aware activation adjustment (arXiv 2509.25689 Sec. 3.2) —
TEST INFRASTRUCTURE ONLY.

Plain-Python statement, for checking the library's host routine.  Only
``tests/`` may import it.

Sec. 3.2: after pruning to a retention ratio r, every layer activates
k_pruned = ceil(r k_orig) experts per token; per device, the per-layer
counts k_i <= k_pruned are tuned so that the per-token active compute
FLOPs_active ~= 2 sum_i k_i P_i (P_i: parameters of one expert of layer i)
fits the device's budget.

Readings where the paper leaves room:
  - ceil is taken as ceil(r k_orig - 1e-12), so that a product that rounding
    lifts just above an integer does not gain an expert;
  - the tuning rule: every layer starts at k_pruned; while FLOPs_active is
    above the budget, one layer loses one activated expert, the layers taken
    in the binary-partition order of Sec. 3.3 (the order its back-off walks
    layers in), cycling through that order, skipping layers already at 1;
  - no layer goes below one expert: if every layer is at 1 and the budget
    still fails, that plan is returned with its (over-budget) FLOPs;
  - topk_group stays as configured: k_i only goes down, so the group rule
    (k_i <= topk_group * E / G) stays satisfiable.
"""
from __future__ import annotations

import math

from oracle.plan import binary_partition_order


def k_pruned(r: float, k_orig: int) -> int:
    return int(math.ceil(r * k_orig - 1e-12))


def flops_active(k_per_layer, params_per_expert) -> int:
    """2 sum_i k_i P_i, exact integers."""
    return 2 * sum(int(k) * int(p) for k, p in zip(k_per_layer, params_per_expert))


def per_layer_k(k_orig: int, r: float, params_per_expert, flops_budget: int):
    """Returns (k_i list, FLOPs_active of that plan)."""
    L = len(params_per_expert)
    kp = k_pruned(r, k_orig)
    k = [kp] * L
    order = binary_partition_order(L)
    pos = 0
    while flops_active(k, params_per_expert) > flops_budget and any(v > 1 for v in k):
        layer = order[pos % L]
        pos += 1
        if k[layer] > 1:
            k[layer] -= 1
    return k, flops_active(k, params_per_expert)
