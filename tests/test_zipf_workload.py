"""The Zipf-skewed prefill workload (config 4) routes like Zipf(1.1): on
token draws other than the one the bias was fitted on (the parity tests'
and the benchmark's), the oracle's routed counts are within L1 0.1 of the
water-filled Zipf(1.1) target over the 192 experts and touch almost all of
them."""
import numpy as np
import pytest

from workloads import get_config
from workloads.synth import draw_router, draw_tokens, zipf_ranks, zipf_target_counts


@pytest.mark.parametrize("token_seed", [101, 1000])
def test_routed_counts_follow_zipf(orc, token_seed):
    spec = get_config("v3_prefill_t2048_zipf")
    T, E, K = spec.tokens, spec.n_experts, spec.top_k
    layer = orc.make_layer(spec.hidden, spec.inter, E, spec.n_groups, spec.topk_group, K, spec.routed_scale,
                           spec.has_shared)
    w, b = draw_router(spec, 0)
    x = draw_tokens(token_seed, T, spec.hidden)
    orc.use_openmp(True)
    try:
        idx, _, _, _ = orc.route(layer, x, w, b)
    finally:
        orc.use_openmp(False)
    counts = np.bincount(idx.reshape(-1), minlength=E)
    target = zipf_target_counts(E, T * K, float(spec.zipf_s), T)[zipf_ranks(spec, 0)]
    l1 = np.abs(counts - target).sum() / (T * K)
    assert l1 <= 0.1, l1
    assert (counts > 0).sum() >= 180
    assert counts.max() <= T


def test_water_filled_target_properties():
    """The target itself: sums to T * k, capped at T, Zipf ratios between
    uncapped ranks."""
    T, E, K, s = 2048, 192, 8, 1.1
    t = zipf_target_counts(E, T * K, s, T)
    assert abs(t.sum() - T * K) < 1e-6
    assert t.max() <= T + 1e-9
    free = t < T - 1e-9
    r = np.arange(1, E + 1)[free]
    np.testing.assert_allclose(t[free] / t[free][0], (r / r[0]) ** (-s), rtol=1e-12)
