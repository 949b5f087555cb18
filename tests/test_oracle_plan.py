"""Pins of the planner oracle (oracle/plan.py) against the paper's own
example and hand-derived cases (arXiv 2509.25689 Sec. 3.3).  No GPU needed."""
import pytest

from oracle import plan as P

# level ladder in 1/64 bit per weight: IQ1_S, IQ1_M, Q2_K, Q3_K, Q4_K, Q5_K, Q6_K, Q8_0
BITS = [100, 112, 168, 220, 288, 352, 420, 544]
IQ1_S, IQ1_M, Q4, Q5, Q6, Q8 = 0, 1, 4, 5, 6, 7
RULES = dict(bits64=BITS, low=IQ1_M, lowest=IQ1_S, small_level=Q8, medium_level=Q6, floor_level=Q4,
             small_max=10_000_000, medium_max=50_000_000)
O, G, U, D = P.KIND_OTHER, P.KIND_GATE, P.KIND_UP, P.KIND_DOWN


def s_low(tensors):
    """S_low in bytes (every test uses parameter counts divisible by 32)."""
    tot = sum(t[0] for t in tensors) * BITS[IQ1_M]
    assert tot % 512 == 0
    return tot // 512


def run(tensors, budget_bytes):
    return P.plan(tensors, mem_limit_bytes=s_low(tensors) + budget_bytes, **RULES)


def _paper(key):
    import json
    import os
    with open(os.path.join(os.path.dirname(__file__), "golden", "paper_examples.json")) as f:
        return json.load(f)[key]


def test_binary_partition_order_paper_example():
    # Sec. 3.3: in a 58-layer MoE the sequence is layer 29, 15, 44, 8, ...
    ex = _paper("binary_partition_order")
    assert P.binary_partition_order(ex["n_layers"])[:len(ex["prefix"])] == ex["prefix"]


@pytest.mark.parametrize("n", list(range(0, 70)) + [128, 255])
def test_binary_partition_order_is_a_permutation(n):
    o = P.binary_partition_order(n)
    assert sorted(o) == list(range(n))


def test_ample_budget_gives_size_class_targets():
    ts = [(5_000_000, 0, O, 0.5), (40_000_000, 0, O, 2.0), (96_000_000, 0, O, 3.0),
          (100_000_000, 1, G, 9.0), (100_000_000, 1, D, 9.0)]
    lv, _ = run(ts, 10 ** 12)
    # < 10M -> Q8, 10M..50M -> Q6, larger stays at Q_low, routed never upgraded
    assert lv == [Q8, Q6, IQ1_M, IQ1_M, IQ1_M]


def test_local_downgrade_one_level():
    # A at Q8 costs 4,218,750 B over Q_low, at Q6 3,007,812.5 B
    ts = [(5_000_000, 0, O, 1.0)]
    assert run(ts, 3_100_000)[0] == [Q6]


def test_local_downgrade_two_levels():
    # Q6 3,007,812.5 B does not fit in 2.5 MB, Q5 2,343,750 B does
    ts = [(5_000_000, 0, O, 1.0)]
    assert run(ts, 2_500_000)[0] == [Q5]


def test_global_downgrade_of_the_largest_earlier_upgrade():
    # B (40M, Q6: 24,062,500 B) first; A (5M) does not fit even at Q5
    # (2,343,750 B of 1,000,000 left); B goes Q6 -> Q5 (18,750,000 B), then
    # A at Q5 fits: 21,093,750 <= 25,062,500
    ts = [(40_000_000, 0, O, 2.0), (5_000_000, 0, O, 1.0)]
    assert run(ts, 24_062_500 + 1_000_000)[0] == [Q5, Q5]


def test_floor_stops_global_downgrade_and_the_tensor_returns_to_low():
    # B fits only at Q4 (13,750,000 B, two local steps); A then finds B at the
    # floor, no routed experts to lower, and stays at Q_low
    ts = [(40_000_000, 0, O, 2.0), (5_000_000, 0, O, 1.0)]
    lv, tot = run(ts, 13_750_000)
    assert lv == [Q4, IQ1_M]
    assert tot <= 512 * (s_low(ts) + 13_750_000)


def test_negative_base_budget_without_routed_experts_upgrades_nothing():
    ts = [(5_000_000, 0, O, 1.0), (8_000_000, 0, O, 2.0)]
    lv, tot = run(ts, -1)
    assert lv == [IQ1_M, IQ1_M]
    assert tot == 512 * s_low(ts)


def test_routed_downgrade_first_layer_in_partition_order():
    # two routed layers (3, 4): the order over positions is 1, 0 -> layer 4;
    # its gate & up free 200M * 12 / 512 = 4,687,500 B, enough for A at Q5
    ts = [(5_000_000, 0, O, 1.0)] + [(100_000_000, ly, k, 0.0) for ly in (3, 4) for k in (G, U, D)]
    lv, _ = run(ts, 2_000_000)
    assert lv == [Q5, IQ1_M, IQ1_M, IQ1_M, IQ1_S, IQ1_S, IQ1_M]


def test_routed_gate_up_of_every_layer_before_any_down():
    # three routed layers: order 2, 1, 0.  A at Q5 needs 15,000,000 B freed:
    # three gate/up steps free 14,062,500, the down of layer 2 another 2,343,750
    ts = [(5_000_000, 0, O, 1.0)] + [(100_000_000, ly, k, 0.0) for ly in (0, 1, 2) for k in (G, U, D)]
    lv, tot = run(ts, 2_343_750 - 15_000_000)
    exp = [Q5] + [IQ1_S, IQ1_S, IQ1_M] * 2 + [IQ1_S, IQ1_S, IQ1_S]
    assert lv == exp
    assert tot <= 512 * (s_low(ts) + 2_343_750 - 15_000_000)


def test_sensitivity_order_and_back_off_sequence():
    # two 5M tensors, room for exactly one at Q8 (4,218,750 B).  The more
    # sensitive one (index 1) takes Q8; index 0 fails at Q8, Q6 and Q5 with
    # nothing left, so the global step lowers index 1: Q8 -> Q6 frees
    # 1,210,937.5 B, Q6 -> Q5 664,062.5 B (1,875,000 B in all, still short of
    # Q5's 2,343,750 B), Q5 -> Q4 625,000 B (2,500,000 B): index 0 fits at Q5
    ts = [(5_000_000, 0, O, 0.1), (5_000_000, 0, O, 0.9)]
    assert run(ts, 4_218_750)[0] == [Q5, Q4]
    # equal sensitivity: the lower index goes first
    ts = [(5_000_000, 0, O, 0.5), (5_000_000, 0, O, 0.5)]
    assert run(ts, 4_218_750)[0] == [Q4, Q5]
    # one byte less: index 0 misses Q8 by a byte and takes Q6 (3,007,812.5 B)
    # in the local step; index 1 then fails at Q8, Q6, Q5 (1,210,936.5 B
    # left), and index 0 goes Q6 -> Q5 (1,874,999 B left) -> Q4 (2,499,999 B
    # left), where index 1 fits at Q5
    lv, tot = run(ts, 4_218_749)
    assert lv == [Q4, Q5]
    assert tot <= 512 * (s_low(ts) + 4_218_749)
