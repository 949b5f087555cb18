"""The layer-stack workload: independent V3-shaped layers (each with its own
mixed-format experts and shared expert) called back to back and captured in
one CUDA graph, as the stack benchmark runs them.  Two full-size layers at
T = 8; the graph replay must give the same bytes as eager calls, and sampled
tokens of every layer match the oracle."""
import numpy as np
import pytest

from tests.gpu_helpers import DeviceLayer, assert_close, mq_lib, tokens
from workloads import get_config
from dataclasses import replace

pytestmark = pytest.mark.gpu


def test_stack_graph_replay_matches_eager_and_oracle(orc):
    import torch
    mq = mq_lib()
    base = get_config("v3_stack20")
    T, L = 8, 2
    spec = replace(base, tokens=T)
    layers = [DeviceLayer(spec, l) for l in range(L)]
    xs = [tokens(spec, 40 + l, T) for l in range(L)]
    xbuf = torch.from_numpy(np.stack(xs).view(np.int16)).cuda()
    outs = torch.full((L, T, spec.hidden), float("nan"), device="cuda")
    idxs = torch.full((L, T, spec.top_k), -1, dtype=torch.int32, device="cuda")
    wts = torch.zeros((L, T, spec.top_k), dtype=torch.float32, device="cuda")
    wsb = mq.moe_quant_workspace_size(layers[0].cfg, T)
    ws = torch.empty(wsb, dtype=torch.uint8, device="cuda")   # shared by the layers (stream-ordered)

    def calls():
        for l, lay in enumerate(layers):
            mq.moe_quant_forward(lay.cfg, T, xbuf[l], lay.router_w, lay.bias, lay.table, lay.fmts, outs[l],
                                 idxs[l], wts[l], ws, wsb)

    stream = torch.cuda.Stream()
    with torch.cuda.stream(stream):
        calls()
    torch.cuda.synchronize()
    eager_out, eager_idx = outs.cpu().numpy().copy(), idxs.cpu().numpy().copy()
    outs.fill_(float("nan"))
    graph = torch.cuda.CUDAGraph()
    with torch.cuda.graph(graph, stream=stream):
        calls()
    graph.replay()
    torch.cuda.synchronize()
    g_out, g_idx = outs.cpu().numpy(), idxs.cpu().numpy()
    np.testing.assert_array_equal(g_idx, eager_idx)
    np.testing.assert_array_equal(g_out.view(np.uint32), eager_out.view(np.uint32))   # deterministic kernels
    for l, lay in enumerate(layers):
        for t in (0, T - 1):
            ry, ridx, _ = lay.oracle_forward(orc, xs[l][t:t + 1], idx_hint=g_idx[l, t])
            np.testing.assert_array_equal(g_idx[l, t:t + 1], ridx)
            assert_close(g_out[l, t:t + 1], ry)


def test_per_layer_k_stack_matches_oracle(orc):
    """Per-layer activated experts (Sec. 3.2): the library's plan for the
    20-layer stack's budget gives k_i in {5, 6}; three V3 layers at k = 6, 5
    and 4 (all <= k_pruned = 6) run back to back, every token of every layer
    against the oracle."""
    mq = mq_lib()
    base = get_config("v3_stack20_ki")
    P = 3 * base.hidden * base.inter
    ex = base.extra
    k, fl = mq.mq_activation_plan(ex["k_orig"], ex["retain"], [P] * base.n_layers,
                                  2 * ex["budget_expert_acts"] * P)
    assert sorted(set(int(v) for v in k)) == [5, 6] and int(k.sum()) == ex["budget_expert_acts"]
    assert fl == 2 * ex["budget_expert_acts"] * P
    T = 5
    for l, kl in enumerate((6, 5, 4)):
        spec = replace(base, tokens=T, top_k=kl)
        lay = DeviceLayer(spec, 60 + l)
        x = tokens(spec, 70 + l, T)
        y, idx, _ = lay.forward(x)
        assert idx.shape == (T, kl)
        ry, ridx, _ = lay.oracle_forward(orc, x, idx_hint=idx)
        np.testing.assert_array_equal(idx, ridx)
        assert_close(y, ry)
