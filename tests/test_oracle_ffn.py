"""Pins for the oracle's expert FFN, combine and shared expert.

The MoE block output is the router-weighted sum of the selected routed
experts' SwiGLU FFNs plus an always-on shared expert (Fig. 1 and the
framework overview of Sec. 3).  The oracle evaluates only the selected
experts, one expert at a time; these tests compare it with a dense numpy
float64 evaluation of EVERY expert on EVERY token followed by selection.
"""
import numpy as np
import pytest

from workloads import get_config
from workloads.synth import (bf16_bits_to_f32, draw_formats, draw_fp32_weights, draw_packed_layer_host,
                             draw_router, draw_tokens, f32_to_bf16_bits)


def _dense_reference(layer, x_bits, Wg, Wu, Wd, idx, wt, shared):
    x = bf16_bits_to_f32(x_bits).astype(np.float64)
    T = x.shape[0]
    y = np.zeros((T, layer.hidden))
    silu = lambda v: v / (1 + np.exp(-v))
    outs = []
    for e in range(len(Wg)):
        g = x @ Wg[e].astype(np.float64).T
        u = x @ Wu[e].astype(np.float64).T
        outs.append((silu(g) * u) @ Wd[e].astype(np.float64).T)   # [T, H]
    for t in range(T):
        for j in range(layer.top_k):
            y[t] += float(wt[t, j]) * outs[idx[t, j]][t]
        if shared:
            y[t] += outs[-1][t]
    return y


def _run(orc, layer, spec_like, x_bits, rw, b, gate, up, down, fmts):
    y, idx, wt = orc.moe_forward(layer, x_bits, rw, b, gate, up, down, fmts)
    n = len(gate)
    Wg = [orc.unpack(fmts[e, 0], gate[e], layer.inter, layer.hidden) for e in range(n)]
    Wu = [orc.unpack(fmts[e, 1], up[e], layer.inter, layer.hidden) for e in range(n)]
    Wd = [orc.unpack(fmts[e, 2], down[e], layer.hidden, layer.inter) for e in range(n)]
    ref = _dense_reference(layer, x_bits, Wg, Wu, Wd, idx, wt, bool(layer.has_shared))
    return y, ref, idx, wt


def test_tiny_layer_matches_dense_brute_force(orc):
    spec = get_config("tiny")
    x = draw_tokens(0, spec.tokens, spec.hidden)
    rw, b = draw_router(spec, 0)
    fmts = draw_formats(spec, 0)
    ws = draw_fp32_weights(spec, 0)
    gate = [orc.pack("Q4_K", g) for g, _, _ in ws]
    up = [orc.pack("Q4_K", u) for _, u, _ in ws]
    down = [orc.pack("Q4_K", d) for _, _, d in ws]
    layer = orc.make_layer(spec.hidden, spec.inter, spec.n_experts, spec.n_groups, spec.topk_group,
                           spec.top_k)
    y, ref, idx, wt = _run(orc, layer, spec, x, rw, b, gate, up, down, fmts)
    assert np.abs(y - ref).max() <= 1e-6 * np.abs(ref).max()
    # the result is the fp32 rounding of the fp64 value
    np.testing.assert_array_equal(y, ref.astype(np.float32))


@pytest.mark.parametrize("seed", [0, 1])
def test_mixed_formats_with_shared_expert(orc, seed):
    """Small layer, every format present, groups on, shared expert."""
    from workloads.configs import LayerSpec
    spec = LayerSpec(name="small_mixed", hidden=256, inter=256, n_experts=8, n_groups=2,
                     topk_group=1, top_k=3, tokens=5, has_shared=True, mixed=True,
                     router_std=1 / 16, bias_std=0.01)
    x = draw_tokens(seed, spec.tokens, spec.hidden)
    rw, b = draw_router(spec, seed)
    fmts = draw_formats(spec, seed)
    fmts[0] = (1, 2, 3)
    fmts[-1] = (4, 4, 4)
    packed = draw_packed_layer_host(spec, seed, fmts)
    n = spec.n_experts + 1
    gate = [packed[e][0] for e in range(n)]
    up = [packed[e][1] for e in range(n)]
    down = [packed[e][2] for e in range(n)]
    layer = orc.make_layer(256, 256, 8, 2, 1, 3, has_shared=True)
    y, ref, idx, wt = _run(orc, layer, spec, x, rw, b, gate, up, down, fmts)
    np.testing.assert_array_equal(y, ref.astype(np.float32))
    # every selected expert lies in the single kept group of its token
    assert all(len(set(int(e) // 4 for e in idx[t])) == 1 for t in range(spec.tokens))


def test_one_hot_token_reproduces_weight_columns(orc):
    """x = e_c: gate/up reduce to column c, so the output is the closed form
    W_d (silu(Wg[:, c]) * Wu[:, c]) for a single expert with weight 1."""
    H, I = 256, 128
    rng = np.random.default_rng(3)
    Wg, Wu, Wd = (rng.normal(0, 0.02, s).astype(np.float32) for s in ((I, H), (I, H), (H, I)))
    pg, pu, pd = orc.pack("Q8_0", Wg), orc.pack("Q8_0", Wu), orc.pack("Q8_0", Wd)
    g, u, d = orc.unpack(4, pg, I, H), orc.unpack(4, pu, I, H), orc.unpack(4, pd, H, I)
    layer = orc.make_layer(H, I, 1, 1, 1, 1)
    for c in (0, 77, 255):
        xf = np.zeros((1, H), np.float32); xf[0, c] = 1.0
        y, idx, wt = orc.moe_forward(layer, f32_to_bf16_bits(xf), np.ones((1, H), np.float32), None,
                                     [pg], [pu], [pd], np.array([[4, 4, 4]], np.uint8))
        assert idx[0, 0] == 0 and wt[0, 0] == 1.0
        gc, uc = g[:, c].astype(np.float64), u[:, c].astype(np.float64)
        h = gc / (1 + np.exp(-gc)) * uc
        want = d.astype(np.float64) @ h
        np.testing.assert_allclose(y[0], want, rtol=1e-6, atol=1e-12)


def test_zero_tokens(orc):
    layer = orc.make_layer(256, 128, 8, 1, 1, 2)
    y, idx, wt = orc.moe_forward(layer, np.zeros((0, 256), np.uint16), np.zeros((8, 256), np.float32),
                                 None, [np.zeros(1, np.uint8)] * 8, [np.zeros(1, np.uint8)] * 8,
                                 [np.zeros(1, np.uint8)] * 8, np.full((8, 3), 3, np.uint8))
    assert y.shape == (0, 256)


def test_openmp_build_gives_identical_bits(orc):
    """The OpenMP build splits rows and tokens over threads without changing
    any row's arithmetic: every output bit equals the single-threaded build's."""
    import os
    spec = get_config("tiny")
    x = draw_tokens(3, 9, spec.hidden)
    rw, b = draw_router(spec, 1)
    fmts = draw_formats(spec, 1)
    ws = draw_fp32_weights(spec, 1)
    gate = [orc.pack("Q4_K", g) for g, _, _ in ws]
    up = [orc.pack("Q4_K", u) for _, u, _ in ws]
    down = [orc.pack("Q4_K", d) for _, _, d in ws]
    layer = orc.make_layer(spec.hidden, spec.inter, spec.n_experts, spec.n_groups, spec.topk_group,
                           spec.top_k)
    y1, idx1, w1 = orc.moe_forward(layer, x, rw, b, gate, up, down, fmts)
    u1 = orc.unpack("Q4_K", gate[0], spec.inter, spec.hidden)
    old = os.environ.get("OMP_NUM_THREADS")
    os.environ["OMP_NUM_THREADS"] = "4"
    try:
        orc.use_openmp(True)
        y2, idx2, w2 = orc.moe_forward(layer, x, rw, b, gate, up, down, fmts)
        u2 = orc.unpack("Q4_K", gate[0], spec.inter, spec.hidden)
    finally:
        orc.use_openmp(False)
        if old is None:
            os.environ.pop("OMP_NUM_THREADS", None)
        else:
            os.environ["OMP_NUM_THREADS"] = old
    np.testing.assert_array_equal(idx1, idx2)
    np.testing.assert_array_equal(w1.view(np.uint32), w2.view(np.uint32))
    np.testing.assert_array_equal(y1.view(np.uint32), y2.view(np.uint32))
    np.testing.assert_array_equal(u1.view(np.uint32), u2.view(np.uint32))
