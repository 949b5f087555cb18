"""Pins for the oracle's router and permutation.

The router scores experts with a sigmoid plus a selection bias, keeps
topk_group groups of the pruned experts and picks num_experts_per_tok
experts (Sec. 3.2, Hardware-Aware Activation Adjustment).  These tests pin
the canonical fp32 arithmetic against exact integer dot products and a
double-precision exp, and the selection against plain top-k and brute
force over all group choices.
"""
import itertools
import math

import numpy as np
import pytest

from workloads.synth import f32_to_bf16_bits, bf16_bits_to_f32


def ulp32(v):
    v = np.float32(abs(v))
    return float(np.spacing(v)) if v > 0 else float(np.spacing(np.float32(0)))


def test_logit_is_exact_integer_dot_product(orc):
    """Small-integer x and W make every product and partial sum exact, so
    the canonical order must return the true dot product: catches a
    transposed or mis-indexed operand."""
    rng = np.random.default_rng(0)
    for H in (128, 256, 1024, 1152, 7168):
        x = rng.integers(-3, 4, H).astype(np.float32)
        w = rng.integers(-5, 6, H).astype(np.float32)
        got = orc.router_logit(f32_to_bf16_bits(x), w)
        assert got == float(np.dot(x.astype(np.int64), w.astype(np.int64)))


def test_logit_close_to_double_dot(orc):
    rng = np.random.default_rng(1)
    H = 7168
    x = f32_to_bf16_bits(rng.standard_normal(H).astype(np.float32))
    w = (rng.standard_normal(H) / math.sqrt(H)).astype(np.float32)
    exact = float(np.dot(bf16_bits_to_f32(x).astype(np.float64), w.astype(np.float64)))
    assert abs(orc.router_logit(x, w) - exact) < 1e-5


def test_sigmoid_special_values(orc):
    assert orc.sigmoid(0.0) == 0.5
    assert orc.sigmoid(100.0) == 1.0
    assert orc.sigmoid(-0.0) == 0.5


def test_sigmoid_within_4_ulp_of_double(orc):
    zs = np.concatenate([np.linspace(-80, 80, 20001), np.linspace(-1, 1, 2001),
                         np.random.default_rng(2).normal(0, 3, 5000)]).astype(np.float32)
    worst = 0.0
    for z in zs:
        got = orc.sigmoid(float(z))
        ref = 1.0 / (1.0 + math.exp(-float(z)))
        worst = max(worst, abs(got - ref) / ulp32(ref))
    assert worst <= 4.0, worst


def _layer(orc, H, E, G, Gk, k, scale=1.0):
    return orc.make_layer(H, 128, E, G, Gk, k, routed_scale=scale)


def _inputs(seed, T, H, E, bias_std=0.01):
    rng = np.random.default_rng(seed)
    x = f32_to_bf16_bits(rng.standard_normal((T, H)).astype(np.float32))
    w = (rng.standard_normal((E, H)) / math.sqrt(H)).astype(np.float32)
    b = (rng.standard_normal(E) * bias_std).astype(np.float32)
    return x, w, b


def _plain_topk(u, k):
    order = sorted(range(len(u)), key=lambda e: (-u[e], e))
    return order[:k]


@pytest.mark.parametrize("E,k", [(8, 2), (64, 6), (192, 8)])
def test_single_group_equals_plain_topk(orc, E, k):
    x, w, b = _inputs(3, 16, 256, E)
    idx, wt, z, s = orc.route(_layer(orc, 256, E, 1, 1, k), x, w, b)
    for t in range(16):
        u = (s[t] + b).astype(np.float32)
        assert list(idx[t]) == _plain_topk(u, k)


def test_all_groups_kept_equals_plain_topk(orc):
    x, w, b = _inputs(4, 16, 256, 192)
    i1, _, _, s = orc.route(_layer(orc, 256, 192, 8, 8, 8), x, w, b)
    i2, _, _, _ = orc.route(_layer(orc, 256, 192, 1, 1, 8), x, w, b)
    np.testing.assert_array_equal(i1, i2)


def test_k_equals_E_selects_all_in_descending_order(orc):
    x, w, b = _inputs(5, 4, 256, 16)
    idx, wt, z, s = orc.route(_layer(orc, 256, 16, 4, 4, 16), x, w, b)
    for t in range(4):
        assert sorted(idx[t]) == list(range(16))
        u = s[t] + b
        assert all(u[idx[t][j]] >= u[idx[t][j + 1]] for j in range(15))


def test_exact_ties_break_to_lower_index(orc):
    """x = 0 gives z = 0 and s = 0.5 for every expert: every group and
    expert ties, so the lowest groups and lowest experts win."""
    H, E = 256, 32
    x = np.zeros((2, H), np.uint16)
    w = np.random.default_rng(6).standard_normal((E, H)).astype(np.float32)
    b = np.zeros(E, np.float32)
    idx, wt, z, s = orc.route(_layer(orc, H, E, 4, 2, 5), x, w, b)
    assert (z == 0).all() and (s == 0.5).all()
    for t in range(2):
        assert list(idx[t]) == [0, 1, 2, 3, 4]
        np.testing.assert_array_equal(wt[t], np.full(5, 0.2, np.float32))


def _brute_force(u, s, E, G, Gk, k):
    gs = E // G
    def gscore(g):
        vals = sorted(u[g * gs:(g + 1) * gs], reverse=True)
        return vals[0] if gs == 1 else np.float32(vals[0]) + np.float32(vals[1])
    best = None
    for groups in itertools.combinations(range(G), Gk):
        tot = sum(float(gscore(g)) for g in groups)
        if best is None or tot > best[0]:
            best = (tot, groups)
    cand = [e for e in range(E) if e // gs in best[1]]
    return sorted(cand, key=lambda e: (-u[e], e))[:k]


@pytest.mark.parametrize("E,G,Gk,k", [(8, 4, 2, 3), (8, 2, 1, 2), (12, 4, 3, 5), (16, 8, 3, 4)])
def test_group_limited_selection_matches_brute_force(orc, E, G, Gk, k):
    x, w, b = _inputs(7 + E + G, 64, 128, E, bias_std=0.05)
    idx, wt, z, s = orc.route(_layer(orc, 128, E, G, Gk, k), x, w, b)
    for t in range(64):
        u = (s[t] + b).astype(np.float32)
        assert list(idx[t]) == _brute_force(u, s[t], E, G, Gk, k)


def test_weights_normalised_and_scaled(orc):
    x, w, b = _inputs(8, 8, 256, 64)
    for scale in (1.0, 2.5):
        idx, wt, z, s = orc.route(_layer(orc, 256, 64, 8, 4, 6, scale), x, w, b)
        for t in range(8):
            sel = s[t][idx[t]].astype(np.float64)
            np.testing.assert_allclose(wt[t], scale * sel / sel.sum(), rtol=3e-7)
            np.testing.assert_allclose(wt[t].sum(), scale, rtol=1e-6)


def test_permutation_invariants(orc):
    rng = np.random.default_rng(9)
    E, T, k = 24, 50, 4
    idx = np.stack([rng.choice(E, k, replace=False) for _ in range(T)]).astype(np.int32)
    off, perm, inv = orc.permute(idx, E)
    counts = np.bincount(idx.reshape(-1), minlength=E)
    np.testing.assert_array_equal(np.diff(off), counts)
    assert off[0] == 0 and off[-1] == T * k
    flat = idx.reshape(-1)
    # sorted by expert, stable (entry ids ascending within an expert)
    for e in range(E):
        seg = perm[off[e]:off[e + 1]]
        assert (flat[seg] == e).all() and (np.diff(seg) > 0).all()
    np.testing.assert_array_equal(perm[inv], np.arange(T * k))
    np.testing.assert_array_equal(inv[perm], np.arange(T * k))


def test_paper_activation_adjustment_and_flops():
    """k_pruned = ceil(r k_orig): r = 0.75, k_orig = 8 gives the deployed 6
    of 192 experts (Sec. 3.2, Sec. 4.1); FLOPs_active = 2 sum k_i P_i."""
    import json
    import os
    from oracle.activation import flops_active
    from oracle.activation import k_pruned as activation_adjusted_k
    with open(os.path.join(os.path.dirname(__file__), "golden", "paper_examples.json")) as f:
        ex = json.load(f)["activation_adjustment"]
    assert activation_adjusted_k(ex["r"], ex["k_orig"]) == ex["k_pruned"]
    assert activation_adjusted_k(0.75, 8) == 6
    from workloads import get_config
    spec = get_config("v3_decode_t1_k6")
    assert spec.top_k == activation_adjusted_k(spec.n_experts / spec.n_original_experts, 8)
    assert activation_adjusted_k(0.75, 256) == 192
    P = 3 * 7168 * 2048
    assert flops_active([8], [P]) == 2 * 8 * P


def test_select_on_precomputed_scores_equals_route(orc):
    """oracle.select re-runs only the selection step: on route's own scores it
    returns route's ids and weights bit for bit, for any bias."""
    from workloads.synth import draw_router, draw_tokens
    from workloads import get_config
    spec = get_config("v3_decode_t1")
    x = draw_tokens(9, 24, spec.hidden)
    rw, b = draw_router(spec, 2)
    layer = orc.make_layer(spec.hidden, spec.inter, spec.n_experts, spec.n_groups, spec.topk_group, spec.top_k)
    for bias in (b, None, b * 40):
        idx, w, z, s = orc.route(layer, x, rw, bias)
        idx2, w2 = orc.select(layer, s, bias)
        np.testing.assert_array_equal(idx, idx2)
        np.testing.assert_array_equal(w.view(np.uint32), w2.view(np.uint32))
