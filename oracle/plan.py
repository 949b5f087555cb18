"""Mixed-precision allocation with back-off (arXiv 2509.25689 Sec. 3.3,
"Hardware-Constrained Budget Formulation" and "Dynamic Allocation with
Back-off") — TEST INFRASTRUCTURE ONLY.

Plain-Python statement of the tensor-level precision planner, written from
the paper's description step by step, for checking the library's planner.
Only ``tests/`` may import it; it shares nothing with the library.

Quantities (Sec. 3.3): every tensor t starts at the base low precision
Q_low; the model then costs S_low.  Upgrading t costs
|t| (b(Q_new, t) - b(Q_low, t)) and downgrading a routed-expert tensor to
Q_low' frees B_delta = |t| (b(Q_low, t) - b(Q_low', t)); a plan is feasible
when the upgrades cost at most B_base + B_delta with B_base = M_limit - S_low,
i.e. when the whole model fits in M_limit.  Costs are counted here in
1/64-bit units per weight (every k-quant width is a multiple of 1/64 bit),
so the budget test is exact integer arithmetic: sum |t| bits64[level_t] <=
512 * M_limit_bytes.

Readings where the paper leaves room (each also listed in the design notes):
  - candidates are the tensors that are not routed-expert tensors, in
    descending Sens(t), ties to the lower input index;
  - size classes: |t| < small_max -> small_level (Q8), small_max <= |t| <=
    medium_max -> medium_level (Q6); larger non-routed tensors stay at Q_low;
    routed-expert tensors are never upgraded;
  - local back-off: the current tensor goes down one level, then a second
    (never below floor_level); if neither fits it keeps the second and the
    global step follows;
  - global back-off: repeatedly, among the tensors upgraded before the
    current one, the one with the most parameters (ties: upgraded earlier)
    that is above floor_level goes down one level (floor_level = Q4: a Q8
    tensor goes down at most three levels, Q8 -> Q6 -> Q5 -> Q4); no back-off
    step takes an upgraded tensor down to Q_low or below;
  - routed back-off: one step per entry of a queue: the gate and up tensors
    of the routed layers in binary-partition order (one step per layer),
    then the down tensors in the same order; each goes from Q_low to Q_low';
  - if the budget still fails after all three, the current tensor returns to
    Q_low (what the earlier steps lowered stays lowered);
  - binary-partition order over n layer positions: the layer at the
    midpoint of the boundaries of [lo, hi), rounded up (clamped to hi - 1),
    then the two halves [lo, mid) and [mid + 1, hi), breadth first — for 58
    layers 29, 15, 44, 8, ... as the paper's example.
"""
from __future__ import annotations

from collections import deque

KIND_OTHER, KIND_GATE, KIND_UP, KIND_DOWN = 0, 1, 2, 3


def binary_partition_order(n: int) -> list[int]:
    out = []
    q = deque([(0, n)])
    while q:
        lo, hi = q.popleft()
        if hi <= lo:
            continue
        mid = min((lo + hi + 1) // 2, hi - 1)
        out.append(mid)
        q.append((lo, mid))
        q.append((mid + 1, hi))
    return out


def plan(tensors, bits64, low, lowest, small_level, medium_level, floor_level, small_max, medium_max,
         mem_limit_bytes):
    """tensors: list of (params, layer, kind, sens).  Returns (levels, total_bits64)."""
    n = len(tensors)
    level = [low] * n
    limit = 512 * mem_limit_bytes

    def total():
        return sum(tensors[i][0] * bits64[level[i]] for i in range(n))

    def fits():
        return total() <= limit

    # routed back-off queue: gate & up per layer, then down per layer
    layers = sorted({t[1] for t in tensors if t[2] != KIND_OTHER})
    order = [layers[p] for p in binary_partition_order(len(layers))]
    queue = []
    for kinds in ((KIND_GATE, KIND_UP), (KIND_DOWN,)):
        for ly in order:
            step = [i for i in range(n) if tensors[i][1] == ly and tensors[i][2] in kinds]
            if step:
                queue.append(step)

    def target(i):
        p = tensors[i][0]
        if p < small_max:
            return small_level
        if p <= medium_max:
            return medium_level
        return low

    cands = [i for i in range(n) if tensors[i][2] == KIND_OTHER and target(i) > low]
    cands.sort(key=lambda i: (-tensors[i][3], i))
    upgraded = []   # in upgrade order
    for i in cands:
        level[i] = target(i)
        if not fits():
            # (1) local downgrade: one level, then a second
            for _ in range(2):
                if level[i] - 1 >= max(floor_level, low + 1):
                    level[i] -= 1
                if fits():
                    break
        if not fits():
            # (2) global large-tensor downgrade among the earlier upgrades
            while not fits():
                best = -1
                for j in upgraded:
                    if level[j] > max(floor_level, low + 1) and (best < 0 or tensors[j][0] > tensors[best][0]):
                        best = j
                if best < 0:
                    break
                level[best] -= 1
        if not fits():
            # (3) routed-expert downgrade in binary-partition layer order
            while not fits() and queue:
                for j in queue.pop(0):
                    level[j] = lowest
        if not fits():
            level[i] = low
            continue
        upgraded.append(i)
    return level, total()
