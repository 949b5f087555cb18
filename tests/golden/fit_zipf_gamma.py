"""Fit the scale gamma of the Zipf bias of the V3 prefill workload.

The prefill workload skews expert counts towards Zipf(1.1) with a per-expert
bias b_e = N(0, 0.01) + gamma * (-1.1 * ln(rank_e + 1)) (rank_e a seeded
permutation).  This script routes a seeded token sample through the oracle
(group-limited selection on) for each candidate gamma and bisects gamma so
that the share of assignments taken by the most popular expert matches the
Zipf(1.1) target, water-filled under the per-token cap of one pick per expert.
It writes tests/golden/zipf_gamma.json; only oracle/ computes routes.

    python tests/golden/fit_zipf_gamma.py
"""
import json
import os
import sys

import numpy as np

ROOT = os.path.dirname(os.path.dirname(os.path.dirname(os.path.abspath(__file__))))
sys.path.insert(0, ROOT)

import oracle  # noqa: E402
from workloads import get_config  # noqa: E402
from workloads.synth import draw_router, draw_tokens, zipf_ranks, zipf_target_counts  # noqa: E402

SAMPLE = 512


def counts_for(spec, layer, x, gamma):
    w, b = draw_router(spec, 0, gamma=gamma)
    idx, _, _, _ = oracle.route(layer, x, w, b)
    ranks = zipf_ranks(spec, 0)
    c = np.bincount(idx.reshape(-1), minlength=spec.n_experts)
    return c[np.argsort(ranks)]   # counts ordered by popularity rank


def main():
    oracle.build()
    spec = get_config("v3_prefill_t2048_zipf")
    layer = oracle.make_layer(spec.hidden, spec.inter, spec.n_experts, spec.n_groups, spec.topk_group, spec.top_k,
                              spec.routed_scale, spec.has_shared)
    x = draw_tokens(4242, SAMPLE, spec.hidden)
    total = SAMPLE * spec.top_k
    target = zipf_target_counts(spec.n_experts, total, float(spec.zipf_s), SAMPLE)
    want = target[0] / total
    lo, hi = 0.0, 1.0
    for _ in range(20):
        mid = 0.5 * (lo + hi)
        share = counts_for(spec, layer, x, mid)[0] / total
        if share < want:
            lo = mid
        else:
            hi = mid
    gamma = 0.5 * (lo + hi)
    got = counts_for(spec, layer, x, gamma)
    l1 = float(np.abs(got - target).sum() / total)
    out = {"gamma": round(gamma, 6), "zipf_s": spec.zipf_s, "tokens_sampled": SAMPLE, "token_seed": 4242,
           "top_share_target": round(float(want), 4), "top_share_got": round(float(got[0] / total), 4),
           "l1_distance_to_target": round(l1, 4),
           "note": "written by tests/golden/fit_zipf_gamma.py (routes computed by oracle/)"}
    with open(os.path.join(ROOT, "tests", "golden", "zipf_gamma.json"), "w") as f:
        json.dump(out, f, indent=2)
    print(json.dumps(out))


if __name__ == "__main__":
    main()
