"""Fit the per-expert selection bias of the V3 prefill workload so that its
routed expert counts follow Zipf(1.1) over the 192 experts.

Target: the Zipf(1.1) shares of the T * k assignments over popularity ranks
(rank_e a seeded permutation of the experts), water-filled under the cap of
T per expert (a token picks an expert at most once).  The bias starts from
the workload's N(0, 0.01) draw and is adjusted on a seeded sample of T
tokens: the logits (and sigmoid scores) do not depend on the bias, so the
oracle routes the sample once and then re-runs only its group-limited
selection for each candidate bias (oracle.select), moving every expert's
bias by a step proportional to log(target / count) until the L1 distance
between the count histogram and the target is small.  The fitted biases are
written, bit-exact (fp32 hex), to tests/golden/zipf_bias.json.  Only oracle/
computes routes.

    python tests/golden/fit_zipf_bias.py
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

TOKEN_SEED = 4242
ITERS = 400


def l1_distance(counts, target, total):
    return float(np.abs(counts - target).sum() / total)


def main():
    oracle.build()
    oracle.use_openmp(True)
    spec = get_config("v3_prefill_t2048_zipf")
    T, E, K = spec.tokens, spec.n_experts, spec.top_k
    layer = oracle.make_layer(spec.hidden, spec.inter, E, spec.n_groups, spec.topk_group, K,
                              spec.routed_scale, spec.has_shared)
    x = draw_tokens(TOKEN_SEED, T, spec.hidden)
    w, b0 = draw_router(spec, 0, base_only=True)
    _, _, _, s = oracle.route(layer, x, w, None)
    ranks = zipf_ranks(spec, 0)
    target = zipf_target_counts(E, T * K, float(spec.zipf_s), T)[ranks]   # per expert id
    bias = b0.astype(np.float64)
    best = (np.inf, None)
    for it in range(ITERS):
        bf = bias.astype(np.float32)
        idx, _ = oracle.select(layer, s, bf)
        counts = np.bincount(idx.reshape(-1), minlength=E).astype(np.float64)
        l1 = l1_distance(counts, target, T * K)
        if l1 < best[0]:
            best = (l1, bf.copy())
        step = 0.05 if it < 150 else (0.02 if it < 300 else 0.008)
        bias += step * (np.log(target + 0.5) - np.log(counts + 0.5))
    l1, bf = best
    idx, _ = oracle.select(layer, s, bf)
    counts = np.bincount(idx.reshape(-1), minlength=E)
    out = {"zipf_s": spec.zipf_s, "tokens_sampled": T, "token_seed": TOKEN_SEED,
           "l1_distance_to_target_on_fit_sample": round(l1, 4),
           "experts_touched_on_fit_sample": int((counts > 0).sum()),
           "top_count_target": float(target.max()), "top_count_got": int(counts.max()),
           "bias_f32_hex": [float(v).hex() for v in bf],
           "note": "written by tests/golden/fit_zipf_bias.py (routes computed by oracle/)"}
    with open(os.path.join(ROOT, "tests", "golden", "zipf_bias.json"), "w") as f:
        json.dump(out, f, indent=1)
    print(json.dumps({k: v for k, v in out.items() if k != "bias_f32_hex"}))


if __name__ == "__main__":
    main()
