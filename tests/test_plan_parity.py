"""The library's planner (mq_plan_precision, mq_binary_partition_order; host
code) against the planner oracle on seeded random models: levels and totals
must be identical (exact integer costs).  No GPU needed."""
import numpy as np
import pytest

from oracle import plan as P
from tests.test_oracle_plan import BITS, IQ1_M, O, G, U, D, Q4, Q8, RULES, s_low


@pytest.fixture(scope="module")
def mq():
    import paper_2509_25689_gb300 as m
    return m


def _random_model(rng):
    n_layers = int(rng.integers(1, 9))
    ts = []
    for ly in range(n_layers):
        for k in (G, U, D):
            if rng.random() < 0.9:
                ts.append((int(rng.integers(1, 4)) * 32 * 1_000_000, ly, k, float(rng.normal())))
        for _ in range(int(rng.integers(0, 6))):
            cls = rng.integers(0, 3)
            p = [int(rng.integers(1, 10_000_000 // 32)) * 32, int(rng.integers(10_000_000 // 32, 50_000_000 // 32 + 1)) * 32,
                 int(rng.integers(50_000_000 // 32 + 1, 80_000_000 // 32)) * 32][cls]
            sens = float(np.round(rng.normal(), 1))   # rounded: ties happen
            ts.append((p, ly, O, sens))
    return ts


@pytest.mark.parametrize("seed", range(60))
def test_library_plan_matches_oracle(mq, seed):
    rng = np.random.default_rng(seed)
    ts = _random_model(rng)
    base = s_low(ts) if ts else 0
    up = sum(t[0] for t in ts if t[2] == O) * (BITS[Q8] - BITS[IQ1_M]) // 512
    for frac in (-0.2, 0.0, 0.05, 0.3, 0.7, 1.2):
        limit = max(0, base + int(frac * up))
        ref_lv, ref_tot = P.plan(ts, mem_limit_bytes=limit, **RULES)
        lv, tot = mq.mq_plan_precision(ts, mem_limit_bytes=limit, **RULES)
        assert list(lv) == ref_lv, (seed, frac)
        assert tot == ref_tot


def test_library_partition_order_matches_oracle(mq):
    for n in list(range(0, 80)) + [58, 256, 1000]:
        assert list(mq.mq_binary_partition_order(n)) == P.binary_partition_order(n)


def test_library_plan_argument_checks(mq):
    ts = [(5_000_000, 0, O, 1.0)]
    with pytest.raises(mq.MoeqError):
        mq.mq_plan_precision(ts, **{**RULES, "bits64": [112, 100]}, mem_limit_bytes=10 ** 9)   # not ascending
    with pytest.raises(mq.MoeqError):
        mq.mq_plan_precision(ts, **{**RULES, "lowest": Q4}, mem_limit_bytes=10 ** 9)        # lowest above low
    with pytest.raises(mq.MoeqError):
        mq.mq_plan_precision([(5, 0, 7, 1.0)], **RULES, mem_limit_bytes=10 ** 9)            # bad kind
    with pytest.raises(mq.MoeqError):
        mq.mq_plan_precision([(5, 0, O, float("nan"))], **RULES, mem_limit_bytes=10 ** 9)   # non-finite
    with pytest.raises(mq.MoeqError):
        mq.mq_plan_precision(ts, **RULES, mem_limit_bytes=-1)
    with pytest.raises(mq.MoeqError):
        mq.mq_binary_partition_order(-1)
    lv, tot = mq.mq_plan_precision([], **RULES, mem_limit_bytes=0)
    assert len(lv) == 0 and tot == 0
