"""Pins of the expert-pruning score oracle (oracle/prune.py, arXiv
2509.25689 Sec. 3.1) with hand-derived values and properties, then the
library's mq_expert_importance against it.  No GPU needed."""
import numpy as np
import pytest

from oracle import prune as R

# three tokens, top-2 of 4 experts, weights exact in binary
IDX = [[0, 1], [0, 2], [0, 1]]
W = [[0.75, 0.25], [0.5, 0.5], [0.625, 0.375]]


def test_hand_example_scores():
    # counts 3, 2, 1, 0 -> f = 1, 2/3, 1/3, 0; weight sums 1.875, 0.625, 0.5
    # -> s = 0.625, 0.3125, 0.5, 0
    s = R.expert_importance(IDX, W, 4, 0.5)
    assert s == [0.5 * 1.0 + 0.5 * 0.625, 0.5 * (2 / 3) + 0.5 * 0.3125, 0.5 * (1 / 3) + 0.5 * 0.5, 0.0]
    assert R.expert_importance(IDX, W, 4, 1.0) == [1.0, 2 / 3, 1 / 3, 0.0]
    assert R.expert_importance(IDX, W, 4, 0.0) == [0.625, 0.3125, 0.5, 0.0]


def test_hand_example_kept_sets():
    # alpha 0.5: I = 0.8125, 0.489..., 0.416..., 0 -> keep {0, 1}
    assert R.prune(IDX, W, 4, 0.5, 0.5)[0] == [0, 1]
    # scores only: expert 2 (mean 0.5) beats expert 1 (mean 0.3125)
    assert R.prune(IDX, W, 4, 0.0, 0.5)[0] == [0, 2]
    # ceil(0.6 * 4) = 3
    assert R.prune(IDX, W, 4, 0.5, 0.6)[0] == [0, 1, 2]


def test_keep_count_is_the_papers_ceiling():
    # Sec. 3.1 keeps ceil(r E): 192 of DeepSeek-V3's 256 routed experts at r = 0.75
    import json
    import os
    with open(os.path.join(os.path.dirname(__file__), "golden", "paper_examples.json")) as f:
        ex = json.load(f)["expert_retention"]
    assert R.keep_count(ex["r"], ex["n_experts"]) == ex["kept"]
    assert R.keep_count(1.0, 256) == 256
    assert R.keep_count(0.001, 256) == 1


def test_ties_keep_the_lower_id():
    idx = [[3, 1], [2, 0]]
    w = [[0.5, 0.5], [0.5, 0.5]]
    # all four experts: f = 1/2, s = 1/2
    assert R.prune(idx, w, 4, 0.5, 0.5)[0] == [0, 1]


@pytest.mark.parametrize("seed", range(5))
def test_frequencies_and_weights_add_up(seed):
    # each token selects top_k distinct experts: sum f_e = top_k; with
    # normalised weights (routed_scale 1) the weight sums add up to n_tokens
    rng = np.random.default_rng(seed)
    T, K, E = 50, 6, 32
    idx = np.stack([rng.choice(E, K, replace=False) for _ in range(T)])
    raw = rng.random((T, K)) + 0.1
    w = (raw / raw.sum(1, keepdims=True)).astype(np.float32)
    f = R.expert_importance(idx, w, E, 1.0)
    assert abs(sum(f) - K) < 1e-12
    counts = np.bincount(idx.reshape(-1), minlength=E)
    s = R.expert_importance(idx, w, E, 0.0)
    assert abs(sum(s[e] * counts[e] for e in range(E)) - T) < 1e-5


def test_never_selected_experts_score_zero_and_go_last():
    idx = [[0, 1]] * 4
    w = [[0.5, 0.5]] * 4
    s = R.expert_importance(idx, w, 5, 0.5)
    assert s[2:] == [0.0, 0.0, 0.0]
    assert R.prune(idx, w, 5, 0.5, 0.6)[0] == [0, 1, 2]


def test_fixed_weight_rounding_by_hand():
    # units of 2^-64, ties to even
    assert R.fixed_weight(1.0) == 2 ** 64
    assert R.fixed_weight(0.625) == 5 * 2 ** 61
    assert R.fixed_weight(2.0 ** -70) == 0              # 1/64 unit
    assert R.fixed_weight(3 * 2.0 ** -66) == 1          # 0.75 unit
    assert R.fixed_weight(2.0 ** -65) == 0              # exactly half: to even (0)
    assert R.fixed_weight(3 * 2.0 ** -65) == 2          # 1.5 units: to even (2)
    assert R.fixed_weight(5 * 2.0 ** -65) == 2          # 2.5 units: to even (2)
    assert R.fixed_weight(-0.75) == -3 * 2 ** 62


def test_weight_sum_is_order_free_and_exact():
    # 1 + 256 * 2^-60: a running double sum loses every small term
    # (1 + 2^-60 rounds back to 1); the exact sum is 1 + 2^-52
    idx = [[0]] * 257
    w = [[1.0]] + [[2.0 ** -60]] * 256
    assert R.expert_importance(idx, w, 1, 0.0) == [(1.0 + 2.0 ** -52) / 257]
    assert R.expert_importance(idx[::-1], w[::-1], 1, 0.0) == [(1.0 + 2.0 ** -52) / 257]


@pytest.mark.parametrize("seed", range(4))
def test_weight_sums_equal_fsum(seed):
    # every float32 weight >= 2^-40 is a whole number of 2^-64 units, so the
    # sum must be the correctly rounded sum of the weights (math.fsum)
    import math
    rng = np.random.default_rng(seed)
    T, K, E = 300, 4, 16
    idx = np.stack([rng.choice(E, K, replace=False) for _ in range(T)])
    w = (rng.random((T, K)) * 2.0 ** rng.integers(-40, 20, (T, K))).astype(np.float32)
    w = np.maximum(w, np.float32(2.0 ** -40))
    count, fsum = R.expert_counts_and_sums(idx.tolist(), w.tolist(), E)
    for e in range(E):
        sel = w[idx == e].astype(np.float64)
        assert count[e] == sel.size
        assert fsum[e] / 2 ** 64 == math.fsum(sel.tolist())


# --------------------------------------------------- library vs the oracle ---
@pytest.fixture(scope="module")
def mq():
    import paper_2509_25689_gb300 as m
    return m


@pytest.mark.parametrize("seed", range(20))
def test_library_matches_oracle(mq, seed):
    rng = np.random.default_rng(100 + seed)
    E = int(rng.integers(8, 257))
    K = int(rng.integers(1, min(E, 9) + 1))
    T = int(rng.integers(1, 400))
    p = rng.zipf(1.3, E).astype(np.float64)
    p /= p.sum()
    idx = np.stack([rng.choice(E, K, replace=False, p=p) for _ in range(T)]).astype(np.int32)
    raw = rng.random((T, K)) + 0.05
    w = (raw / raw.sum(1, keepdims=True) * (2.5 if seed % 2 else 1.0)).astype(np.float32)
    for alpha, r in ((0.5, 0.75), (0.0, 0.5), (1.0, 0.3), (0.25, 1.0)):
        keep, scores = mq.mq_expert_importance(idx, w, E, alpha, r)
        rkeep, rscores = R.prune(idx.tolist(), w.tolist(), E, alpha, r)
        assert list(keep) == rkeep
        np.testing.assert_array_equal(scores, np.array(rscores))


def test_library_argument_checks(mq):
    idx = np.zeros((2, 2), np.int32)
    w = np.ones((2, 2), np.float32)
    for bad in (dict(alpha=1.5), dict(alpha=-0.1), dict(retain=0.0), dict(retain=1.1)):
        with pytest.raises(mq.MoeqError):
            mq.mq_expert_importance(idx, w, 4, **bad)
    with pytest.raises(mq.MoeqError):
        mq.mq_expert_importance(np.full((2, 2), 4, np.int32), w, 4)      # id out of range
    with pytest.raises(mq.MoeqError):
        mq.mq_expert_importance(idx, np.full((2, 2), np.nan, np.float32), 4)
    keep, scores = mq.mq_expert_importance(np.zeros((0, 2), np.int32), np.zeros((0, 2), np.float32), 4, 0.5, 0.5)
    assert list(keep) == [0, 1] and (scores == 0).all()


def test_library_exact_sums_hard_weights(mq):
    # weights over 2^-80 .. 2^31, negatives, zeros, and 1 + 256 * 2^-60 on one
    # expert: the host routine's fixed-point sums give the oracle's bits
    rng = np.random.default_rng(5)
    E, K, T = 40, 4, 800
    idx = np.stack([rng.choice(E, K, replace=False) for _ in range(T)]).astype(np.int32)
    w = (rng.random((T, K)) * 2.0 ** rng.integers(-80, 31, (T, K))).astype(np.float32)
    w[rng.random((T, K)) < 0.1] *= -1
    w[rng.random((T, K)) < 0.05] = 0.0
    idx[:257, 0] = 3
    w[:257, 0] = np.float32(2.0 ** -60)
    w[0, 0] = np.float32(1.0)
    for alpha, r in ((0.5, 0.75), (0.0, 0.5)):
        keep, scores = mq.mq_expert_importance(idx, w, E, alpha, r)
        rkeep, rscores = R.prune(idx.tolist(), w.tolist(), E, alpha, r)
        assert list(keep) == rkeep
        np.testing.assert_array_equal(scores.view(np.uint64), np.array(rscores).view(np.uint64))
    with pytest.raises(mq.MoeqError):      # |w| >= 2^32 is outside the accumulator's range
        mq.mq_expert_importance(idx[:1], np.full((1, K), 2.0 ** 32, np.float32), E)


def test_device_stats_host_side_checks(mq):
    # sizes and argument checks that reject (or finish) before any device work
    assert mq.mq_expert_stats_bytes(0) == 0 and mq.mq_expert_stats_bytes(1025) == 0
    assert mq.mq_expert_stats_bytes(256) == 16 + 24 * 256
    buf = np.zeros(mq.mq_expert_stats_bytes(256) + 16, np.uint8)
    base = buf.ctypes.data
    stats = base + (-base) % 16
    assert mq.mq_expert_stats_add(stats, 256, None, None, 0, 8) == 0          # empty batch: nothing enqueued
    for r, k in ((0.75, 192), (1.0, 256), (0.5, 128), (0.001, 1)):
        assert mq.mq_expert_stats_scores(stats, 256, 0.5, r) == k == R.keep_count(r, 256)
    with pytest.raises(mq.MoeqError):
        mq.mq_expert_stats_reset(stats, 0)
    with pytest.raises(mq.MoeqError):
        mq.mq_expert_stats_scores(stats, 256, 1.5, 0.75)
    with pytest.raises(mq.MoeqError):
        mq.mq_expert_stats_scores(stats, 256, 0.5, 0.0)
    with pytest.raises(mq.MoeqError):
        mq.mq_expert_stats_add(stats, 256, None, None, 4, 8)                 # null batch
    with pytest.raises(mq.MoeqError):
        mq.mq_expert_stats_add(stats, 256, 16, 16, 4, 33)                    # top_k > 32
    with pytest.raises(mq.MoeqError):
        mq.mq_expert_stats_add(stats + 8, 256, 16, 16, 4, 8)                 # misaligned buffer
