"""Pins of the activation-adjustment oracle (oracle/activation.py, arXiv
2509.25689 Sec. 3.2) with hand-derived plans, then the library's
mq_activation_plan against it.  No GPU needed."""
import json
import os

import numpy as np
import pytest

from oracle import activation as A

P_V3 = 3 * 7168 * 2048          # parameters of one V3 routed expert (gate, up, down)


def test_k_pruned_is_the_papers_value():
    with open(os.path.join(os.path.dirname(__file__), "golden", "paper_examples.json")) as f:
        ex = json.load(f)["activation_adjustment"]
    assert A.k_pruned(ex["r"], ex["k_orig"]) == ex["k_pruned"] == 6
    assert A.k_pruned(1.0, 8) == 8
    assert A.k_pruned(0.5, 8) == 4
    assert A.k_pruned(0.3, 8) == 3          # 2.4 -> 3
    assert A.k_pruned(0.01, 8) == 1


def test_flops_active_formula():
    # 2 sum k_i P_i
    assert A.flops_active([6, 5], [10, 20]) == 2 * (60 + 100)
    assert A.flops_active([8] * 58, [P_V3] * 58) == 2 * 8 * 58 * P_V3


def test_budget_met_at_k_pruned_changes_nothing():
    k, f = A.per_layer_k(8, 0.75, [P_V3] * 20, 2 * 6 * 20 * P_V3)
    assert k == [6] * 20 and f == 2 * 120 * P_V3


def test_hand_plan_four_layers():
    # binary-partition order of 4 layers: 2 (midpoint of [0,4)), 1 ([0,2)),
    # 3 ([3,4)), 0 ([0,1)).  k_pruned = ceil(0.75 * 8) = 6, P = 1:
    # 24 at k_pruned; budget 2 * 21 -> three layers lose one, in that order
    k, f = A.per_layer_k(8, 0.75, [1, 1, 1, 1], 42)
    assert k == [6, 5, 5, 5] and f == 42
    # budget 2 * 17: seven steps: 2, 1, 3, 0, 2, 1, 3
    k, f = A.per_layer_k(8, 0.75, [1, 1, 1, 1], 34)
    assert k == [5, 4, 4, 4] and f == 34
    # odd budget: stop at the first plan at or below it
    k, f = A.per_layer_k(8, 0.75, [1, 1, 1, 1], 43)
    assert k == [6, 5, 5, 5] and f == 42


def test_hand_plan_unequal_experts():
    # P = [10, 1, 1]: order of 3 layers is 2 ([0,3) midpoint rounded up... (0+3+1)//2 = 2),
    # then [0,2) -> 1, then [0,1) -> 0.  k_pruned 2 (r 0.5, k_orig 4).
    # start 2 * (20 + 2 + 2) = 48; budget 40: layer 2 -> 46, layer 1 -> 44,
    # layer 0 -> 24 (fits)
    k, f = A.per_layer_k(4, 0.5, [10, 1, 1], 40)
    assert k == [1, 1, 1] and f == 24
    k, f = A.per_layer_k(4, 0.5, [10, 1, 1], 47)
    assert k == [2, 2, 1] and f == 46


def test_floor_of_one_expert():
    k, f = A.per_layer_k(8, 0.75, [5, 5], 1)
    assert k == [1, 1] and f == 20


def test_58_layers_start_with_the_papers_partition_prefix():
    # budget one expert short of k_pruned everywhere: only layer 29 (the first
    # of the order 29, 15, 44, 8, ...) gives one up
    k, _ = A.per_layer_k(8, 0.75, [P_V3] * 58, 2 * (6 * 58 - 1) * P_V3)
    assert [i for i in range(58) if k[i] == 5] == [29]
    k, _ = A.per_layer_k(8, 0.75, [P_V3] * 58, 2 * (6 * 58 - 4) * P_V3)
    assert sorted(i for i in range(58) if k[i] == 5) == [8, 15, 29, 44]


# --------------------------------------------------- library vs the oracle ---
@pytest.fixture(scope="module")
def mq():
    import paper_2509_25689_gb300 as m
    return m


@pytest.mark.parametrize("seed", range(30))
def test_library_matches_oracle(mq, seed):
    rng = np.random.default_rng(300 + seed)
    L = int(rng.integers(1, 70))
    k_orig = int(rng.integers(1, 17))
    r = float(rng.choice([0.25, 0.5, 0.6, 0.75, 0.9, 1.0]))
    P = [int(v) for v in rng.integers(1, 1 << 30, L)]
    full = A.flops_active([A.k_pruned(r, k_orig)] * L, P)
    budget = int(rng.integers(0, full + 2))
    k, f = mq.mq_activation_plan(k_orig, r, P, budget)
    rk, rf = A.per_layer_k(k_orig, r, P, budget)
    assert list(k) == rk and f == rf


def test_library_argument_checks(mq):
    for bad in (dict(k_orig=0), dict(retain=0.0), dict(retain=1.5), dict(budget=-1), dict(P=[0]),
                dict(P=[1 << 41])):
        args = dict(k_orig=8, retain=0.75, P=[100], budget=1000)
        args.update(bad)
        with pytest.raises(mq.MoeqError):
            mq.mq_activation_plan(args["k_orig"], args["retain"], args["P"], args["budget"])
    k, f = mq.mq_activation_plan(8, 0.75, [], 0)
    assert list(k) == [] and f == 0
