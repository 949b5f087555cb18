"""GPU parity: the CUDA path through the C ABI vs the oracle on the same
seeded inputs.  Bit-exact for unpacked weights, expert ids, routing weights
and the permutation; max |err| <= 2e-3 * max|y| for the layer output."""
from dataclasses import replace

import numpy as np
import pytest

from tests.gpu_helpers import DeviceLayer, assert_close, mq_lib, tokens
from workloads import get_config
from workloads.configs import LayerSpec
from workloads.synth import random_packed, rng_for

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def torch_cuda():
    import torch
    assert torch.cuda.is_available()
    return torch


# ---------------------------------------------------------------- unpack ---
@pytest.mark.parametrize("fmt", [1, 2, 3, 4])
@pytest.mark.parametrize("shape", [(16, 256), (33, 300), (128, 7168), (7168, 2048)])
def test_unpack_device_bit_exact(torch_cuda, orc, fmt, shape):
    mq = mq_lib()
    rows, cols = shape
    p = random_packed(fmt, rows, cols, rng_for(fmt * 31 + rows))
    dev = torch_cuda.from_numpy(p).cuda()
    out = torch_cuda.empty((rows, cols), dtype=torch_cuda.float32, device="cuda")
    mq.mq_unpack_device(fmt, dev, rows, cols, out)
    got = out.cpu().numpy()
    ref = orc.unpack(fmt, p, rows, cols)
    np.testing.assert_array_equal(got.view(np.uint32), ref.view(np.uint32))


# --------------------------------------------------------------- routing ---
def _route(torch, layer: DeviceLayer, x_bits):
    mq = mq_lib()
    T, K, E = x_bits.shape[0], layer.spec.top_k, layer.spec.n_experts
    x = torch.from_numpy(np.ascontiguousarray(x_bits).view(np.int16)).cuda()
    idx = torch.full((T, K), -1, dtype=torch.int32, device="cuda")
    w = torch.zeros((T, K), dtype=torch.float32, device="cuda")
    off = torch.zeros(E + 1, dtype=torch.int32, device="cuda")
    perm = torch.zeros(max(T * K, 1), dtype=torch.int32, device="cuda")
    inv = torch.zeros(max(T * K, 1), dtype=torch.int32, device="cuda")
    wsb = mq.moe_quant_workspace_size(layer.cfg, T)
    ws = torch.empty(wsb, dtype=torch.uint8, device="cuda")
    mq.moe_quant_route(layer.cfg, T, x, layer.router_w, layer.bias, idx, w, off, perm, inv, ws, wsb)
    torch.cuda.synchronize()
    return idx.cpu().numpy(), w.cpu().numpy(), off.cpu().numpy(), perm.cpu().numpy()[:T * K], inv.cpu().numpy()[:T * K]


class _RouterOnly:
    """Router inputs of a config without allocating expert tensors."""

    def __init__(self, spec, seed):
        import torch
        from workloads.synth import draw_router
        mq = mq_lib()
        self.spec = spec
        rw, b = draw_router(spec, seed)
        self.router_w_host, self.bias_host = rw, b
        self.router_w, self.bias = torch.from_numpy(rw).cuda(), torch.from_numpy(b).cuda()
        self.cfg = mq.make_cfg(spec.hidden, spec.inter, spec.n_experts, spec.n_groups, spec.topk_group,
                               spec.top_k, spec.routed_scale, spec.has_shared)


@pytest.mark.parametrize("name,T", [("tiny", 4), ("tiny", 1), ("v3_decode_t1", 1), ("v3_decode_t1", 7),
                                    ("v3_decode_t1_k6", 1), ("v3_decode_t1_k6", 5),
                                    ("v3_decode_t32_mixed", 32), ("v3_decode_t32_mixed", 256),
                                    ("v3_decode_t32_mixed", 257), ("v3_prefill_t2048_zipf", 2048)])
def test_routing_bit_exact(torch_cuda, orc, name, T):
    spec = get_config(name)
    lay = _RouterOnly(spec, 0)
    x = tokens(spec, 0, T)
    idx, w, off, perm, inv = _route(torch_cuda, lay, x)
    layer = orc.make_layer(spec.hidden, spec.inter, spec.n_experts, spec.n_groups, spec.topk_group, spec.top_k,
                           spec.routed_scale, spec.has_shared)
    ridx, rw, _, _ = orc.route(layer, x, lay.router_w_host, lay.bias_host)
    np.testing.assert_array_equal(idx, ridx)
    np.testing.assert_array_equal(w.view(np.uint32), rw.view(np.uint32))
    roff, rperm, rinv = orc.permute(ridx, spec.n_experts)
    np.testing.assert_array_equal(off, roff)
    np.testing.assert_array_equal(perm, rperm)
    np.testing.assert_array_equal(inv, rinv)


MAX_ROUTER = LayerSpec(name="max_router", hidden=256, inter=256, n_experts=256, n_groups=64, topk_group=16,
                       top_k=32, tokens=1, has_shared=True, mixed=True, router_std=1 / 16, bias_std=0.01)


@pytest.mark.parametrize("T", [1, 3, 300])
def test_routing_bit_exact_largest_shapes(torch_cuda, orc, T):
    """256 experts, 64 groups of 4, top-32: every lane holds a selection in
    the one-token path, the group scan takes its lane-per-group form, and
    T = 300 goes through the separate top-k and permutation kernels."""
    spec = replace(MAX_ROUTER, tokens=T)
    lay = _RouterOnly(spec, 2)
    x = tokens(spec, 2, T)
    idx, w, off, perm, inv = _route(torch_cuda, lay, x)
    layer = orc.make_layer(spec.hidden, spec.inter, spec.n_experts, spec.n_groups, spec.topk_group, spec.top_k,
                           spec.routed_scale, spec.has_shared)
    ridx, rw, _, _ = orc.route(layer, x, lay.router_w_host, lay.bias_host)
    np.testing.assert_array_equal(idx, ridx)
    np.testing.assert_array_equal(w.view(np.uint32), rw.view(np.uint32))
    roff, rperm, rinv = orc.permute(ridx, spec.n_experts)
    np.testing.assert_array_equal(off, roff)
    np.testing.assert_array_equal(perm, rperm)
    np.testing.assert_array_equal(inv, rinv)


@pytest.mark.parametrize("T", [1, 40])
def test_routing_bit_exact_largest_hidden(torch_cuda, orc, T):
    """Hidden 32768 (the largest accepted): 32 segments of 1024 per logit, so
    the per-expert logits kernel runs with 32 warps, also for 40 tokens (the
    tiled kernel takes at most 8 segments)."""
    spec = LayerSpec(name="wide_router", hidden=32768, inter=128, n_experts=16, n_groups=4, topk_group=2,
                     top_k=4, tokens=T, has_shared=False, router_std=1 / 181.0, bias_std=0.01)
    lay = _RouterOnly(spec, 3)
    x = tokens(spec, 3, T)
    idx, w, off, perm, inv = _route(torch_cuda, lay, x)
    layer = orc.make_layer(spec.hidden, spec.inter, spec.n_experts, spec.n_groups, spec.topk_group, spec.top_k,
                           spec.routed_scale, spec.has_shared)
    ridx, rw, _, _ = orc.route(layer, x, lay.router_w_host, lay.bias_host)
    np.testing.assert_array_equal(idx, ridx)
    np.testing.assert_array_equal(w.view(np.uint32), rw.view(np.uint32))
    roff, rperm, rinv = orc.permute(ridx, spec.n_experts)
    np.testing.assert_array_equal(off, roff)
    np.testing.assert_array_equal(perm, rperm)


@pytest.mark.parametrize("T", [1, 3])
def test_forward_largest_routing_shapes(torch_cuda, orc, T, decode_kernel):
    """Top-32 of 256 mixed-format experts plus the shared one: 33 slots per
    token through the decode kernels."""
    spec = replace(MAX_ROUTER, tokens=T)
    layer = DeviceLayer(spec, 5)
    x = tokens(spec, 5, T)
    y, idx, w = layer.forward(x)
    ry, ridx, rw = layer.oracle_forward(orc, x, idx_hint=idx)
    np.testing.assert_array_equal(idx, ridx)
    assert_close(y, ry)


@pytest.mark.parametrize("hidden", [256, 768, 1280])
def test_forward_one_token_shared_k_halves(torch_cuda, orc, hidden):
    """One token: the shared expert's gate/up blocks are split in two K halves
    (K = hidden) whose sums the second-finishing half adds.  1, 3 and 5
    superblocks: no split, then unequal halves."""
    mq = mq_lib()
    spec = LayerSpec(name="k_halves", hidden=hidden, inter=256, n_experts=12, n_groups=4, topk_group=2, top_k=3,
                     tokens=1, has_shared=True, mixed=True, router_std=1 / hidden ** 0.5, bias_std=0.01)
    fm = np.array([[1, 2, 3], [2, 3, 4], [3, 4, 1], [4, 1, 2]] * 3 + [[4, 4, 4]], np.uint8)
    layer = DeviceLayer(spec, hidden, fmts=fm)
    x = tokens(spec, hidden)
    mq.mq_set_path(1)
    try:
        y, idx, w = layer.forward(x)
    finally:
        mq.mq_set_path(0)
    ry, ridx, rw = layer.oracle_forward(orc, x)
    np.testing.assert_array_equal(idx, ridx)
    assert_close(y, ry)


@pytest.mark.parametrize("T", [1, 3])
def test_forward_sizes_not_multiple_of_256(torch_cuda, orc, T, decode_kernel):
    """Hidden 384 and inter 128 (multiples of 128 only) with every format,
    Q8_0 included: these shapes always take the tcgen05 decode kernels (the
    mma.sync ones stream whole 256-element superblocks)."""
    spec = LayerSpec(name="odd_sizes", hidden=384, inter=128, n_experts=12, n_groups=4, topk_group=2, top_k=3,
                     tokens=T, has_shared=True, mixed=True, router_std=1 / 19.6, bias_std=0.01)
    fm = np.array([[1, 2, 3], [2, 3, 4], [3, 4, 1], [4, 1, 2]] * 3 + [[4, 4, 4]], np.uint8)
    layer = DeviceLayer(spec, T, fmts=fm)
    x = tokens(spec, T)
    y, idx, w = layer.forward(x)
    ry, ridx, rw = layer.oracle_forward(orc, x)
    np.testing.assert_array_equal(idx, ridx)
    assert_close(y, ry)


def test_expert_pruning_scores_from_device_routing(torch_cuda, orc):
    """Sec. 3.1 on the unpruned router (256 experts, 8 groups, top-8): a
    synthetic calibration stream routed on the GPU, the importance scores and
    the kept 192 experts from the library's host routine, against the oracle
    routing the same tokens and scoring them itself."""
    from oracle import prune as R
    mq = mq_lib()
    spec = LayerSpec(name="v3_unpruned_router", hidden=7168, inter=2048, n_experts=256, n_groups=8, topk_group=4,
                     top_k=8, tokens=512, has_shared=True, router_std=1 / 7168 ** 0.5, bias_std=0.01)
    lay = _RouterOnly(spec, 4)
    x = tokens(spec, 4, 512)
    idx, w, *_ = _route(torch_cuda, lay, x)
    keep, scores = mq.mq_expert_importance(idx, w, 256, 0.5, 0.75)
    layer = orc.make_layer(spec.hidden, spec.inter, spec.n_experts, spec.n_groups, spec.topk_group, spec.top_k,
                           spec.routed_scale, spec.has_shared)
    ridx, rw, _, _ = orc.route(layer, x, lay.router_w_host, lay.bias_host)
    rkeep, rscores = R.prune(ridx.tolist(), rw.tolist(), 256, 0.5, 0.75)
    assert len(keep) == 192
    assert list(keep) == rkeep
    np.testing.assert_array_equal(scores, np.array(rscores))


@pytest.mark.parametrize("T", [1, 3])
def test_routing_tie_break_on_device(torch_cuda, orc, T):
    """All-zero activations tie every expert; lowest ids must win (one token
    takes the one-warp routing path, three the per-warp one)."""
    spec = LayerSpec(name="ties", hidden=256, inter=128, n_experts=32, n_groups=4, topk_group=2, top_k=5,
                     tokens=T, has_shared=False, router_std=0.1, bias_std=0.0)
    lay = _RouterOnly(spec, 1)
    x = np.zeros((T, 256), np.uint16)
    idx, w, *_ = _route(torch_cuda, lay, x)
    assert (idx == np.arange(5)).all()
    assert (w == np.float32(0.2)).all()


# --------------------------------------------------------------- forward ---
@pytest.fixture(params=[1, 3], ids=["mma", "tc"])
def decode_kernel(request):
    """Decode path on the mma.sync GEMV kernels (1) or the tcgen05 ones (3)."""
    mq = mq_lib()
    mq.mq_set_path(request.param)
    yield request.param
    mq.mq_set_path(0)


def test_forward_tiny_layer(torch_cuda, orc, decode_kernel):
    spec = get_config("tiny")
    layer = DeviceLayer(spec, 0, orc=orc)
    x = tokens(spec, 0)
    y, idx, w = layer.forward(x)
    ry, ridx, rw = layer.oracle_forward(orc, x)
    np.testing.assert_array_equal(idx, ridx)
    np.testing.assert_array_equal(w.view(np.uint32), rw.view(np.uint32))
    assert_close(y, ry)


def test_forward_tiny_layer_one_token_no_shared(torch_cuda, orc, decode_kernel):
    """One token and no shared expert: the one-warp routing path (no block-wide
    sort) and the one-token FFN kernels with routed slots only."""
    spec = get_config("tiny")
    assert not spec.has_shared
    layer = DeviceLayer(spec, 0, orc=orc)
    x = tokens(spec, 0, 1)
    y, idx, w = layer.forward(x)
    ry, ridx, rw = layer.oracle_forward(orc, x)
    np.testing.assert_array_equal(idx, ridx)
    np.testing.assert_array_equal(w.view(np.uint32), rw.view(np.uint32))
    assert_close(y, ry)


SMALL_MIXED = LayerSpec(name="small_mixed", hidden=512, inter=256, n_experts=12, n_groups=4, topk_group=2,
                        top_k=3, tokens=1, has_shared=True, mixed=True, router_std=1 / 22.6, bias_std=0.01)
SMALL_MIXED_FMTS = np.array([[1, 2, 3], [2, 3, 4], [3, 4, 1], [4, 1, 2]] * 3 + [[4, 4, 4]], np.uint8)


@pytest.mark.parametrize("T", [1, 3, 5, 9, 40, 63])
def test_forward_small_mixed_layer_with_shared(torch_cuda, orc, T, decode_kernel):
    spec = replace(SMALL_MIXED, tokens=T)
    layer = DeviceLayer(spec, T, fmts=SMALL_MIXED_FMTS)
    x = tokens(spec, T)
    y, idx, w = layer.forward(x)
    ry, ridx, rw = layer.oracle_forward(orc, x)
    np.testing.assert_array_equal(idx, ridx)
    assert_close(y, ry)


@pytest.mark.parametrize("T", [1, 6])
def test_forward_routed_scale(torch_cuda, orc, T, decode_kernel):
    """routed_scale != 1 (Sec. 3.2 weights scaled after normalisation): the
    weights stay bit-exact and the output follows them."""
    spec = replace(SMALL_MIXED, tokens=T, routed_scale=2.5)
    layer = DeviceLayer(spec, 11 + T, fmts=SMALL_MIXED_FMTS)
    x = tokens(spec, 11 + T)
    y, idx, w = layer.forward(x)
    ry, ridx, rw = layer.oracle_forward(orc, x)
    np.testing.assert_array_equal(idx, ridx)
    np.testing.assert_array_equal(w.view(np.uint32), rw.view(np.uint32))
    assert_close(y, ry)


def test_forward_decode_beyond_cached_assignments(torch_cuda, orc, decode_kernel):
    """2,400 routed assignments on the decode kernels, more than either keeps
    in shared memory: the rest come from the permutation in global memory."""
    spec = LayerSpec(name="many_assign", hidden=256, inter=256, n_experts=64, n_groups=8, topk_group=4,
                     top_k=8, tokens=300, has_shared=True, mixed=True, router_std=1 / 16, bias_std=0.01)
    layer = DeviceLayer(spec, 5)
    x = tokens(spec, 5)
    y, idx, w = layer.forward(x)
    ry, ridx, rw = layer.oracle_forward(orc, x)
    np.testing.assert_array_equal(idx, ridx)
    np.testing.assert_array_equal(w.view(np.uint32), rw.view(np.uint32))
    assert_close(y, ry)


def test_forward_v3_decode_t1(torch_cuda, orc, decode_kernel):
    spec = get_config("v3_decode_t1")
    layer = DeviceLayer(spec, 0)
    x = tokens(spec, 0)
    y, idx, w = layer.forward(x)
    ry, ridx, rw = layer.oracle_forward(orc, x, idx_hint=idx)
    np.testing.assert_array_equal(idx, ridx)
    assert_close(y, ry)


@pytest.mark.parametrize("T", [1, 5])
def test_forward_v3_decode_k6(torch_cuda, orc, T, decode_kernel):
    """The activation-adjusted layer (k = 6 of 192, Sec. 3.2) on the same kernels."""
    spec = get_config("v3_decode_t1_k6")
    layer = DeviceLayer(spec, 2)
    x = tokens(spec, 2, T)
    y, idx, w = layer.forward(x)
    for t in sorted({0, T - 1}):
        ry, ridx, rw = layer.oracle_forward(orc, x[t:t + 1], idx_hint=idx[t])
        np.testing.assert_array_equal(idx[t:t + 1], ridx)
        np.testing.assert_array_equal(w[t:t + 1].view(np.uint32), rw.view(np.uint32))
        assert_close(y[t:t + 1], ry)


def test_forward_v3_decode_t32_mixed_full(torch_cuda, orc, decode_kernel):
    """Config 3 in full: all 32 tokens of the mixed-format V3 layer against one
    oracle call (the oracle's OpenMP build, identical bits to the plain one)."""
    spec = get_config("v3_decode_t32_mixed")
    layer = DeviceLayer(spec, 0)
    x = tokens(spec, 0)
    y, idx, w = layer.forward(x)
    orc.use_openmp(True)
    try:
        ry, ridx, rw = layer.oracle_forward(orc, x, idx_hint=idx)
    finally:
        orc.use_openmp(False)
    np.testing.assert_array_equal(idx, ridx)
    np.testing.assert_array_equal(w.view(np.uint32), rw.view(np.uint32))
    assert_close(y, ry)
    for t in range(spec.tokens):   # and every token against its own scale
        assert_close(y[t:t + 1], ry[t:t + 1])


def test_status_word_clean_after_forward_on_every_path(torch_cuda):
    """The error word the kernels set when a bounded wait gives up stays 0 on
    normal calls, on the decode (both kernels) and prefill paths."""
    import torch
    mq = mq_lib()
    spec = replace(SMALL_MIXED, tokens=5)
    layer = DeviceLayer(spec, 3, fmts=SMALL_MIXED_FMTS)
    T = 5
    x = torch.from_numpy(tokens(spec, 3).view(np.int16)).cuda()
    out = torch.empty((T, spec.hidden), device="cuda")
    wsb = mq.moe_quant_workspace_size(layer.cfg, T)
    ws = torch.empty(wsb, dtype=torch.uint8, device="cuda")
    for path in (1, 2, 3):
        mq.mq_set_path(path)
        try:
            mq.moe_quant_forward(layer.cfg, T, x, layer.router_w, layer.bias, layer.table, layer.fmts, out,
                                 workspace=ws, ws_bytes=wsb)
        finally:
            mq.mq_set_path(0)
        assert mq.moe_quant_status(layer.cfg, T, ws, wsb) == 0
        assert torch.isfinite(out).all()


@pytest.mark.parametrize("T", [1, 3])
def test_wait_give_up_reports_status_and_context_stays_usable(torch_cuda, orc, T):
    """The bounded-wait give-up path, made to run out on purpose: a test hook
    shortens every pipeline wait of the next decode call to 1 ms and has the
    gate/up producer post nothing for its first stage.  The consumers' wait
    on that stage ends, the kernels record it in the error word and exit
    (no copy left in flight), moe_quant_status returns MQ_EDEVICE with the
    full-barrier bit, and the next call runs normally and matches the oracle.
    T = 1 runs the one-token kernel, whose item-finishing warp then has to
    leave its wait for items that never come; T = 3 the several-token one."""
    import torch
    mq = mq_lib()
    spec = replace(SMALL_MIXED, tokens=T)
    layer = DeviceLayer(spec, 4, fmts=SMALL_MIXED_FMTS)
    x_bits = tokens(spec, 4)
    x = torch.from_numpy(x_bits.view(np.int16)).cuda()
    out = torch.empty((T, spec.hidden), device="cuda")
    wsb = mq.moe_quant_workspace_size(layer.cfg, T)
    ws = torch.empty(wsb, dtype=torch.uint8, device="cuda")
    mq.mq_set_path(1)
    try:
        mq.mq_test_fail_next_decode(1_000_000)
        mq.moe_quant_forward(layer.cfg, T, x, layer.router_w, layer.bias, layer.table, layer.fmts, out,
                             workspace=ws, ws_bytes=wsb)
        bits = mq.moe_quant_status(layer.cfg, T, ws, wsb)
        assert bits & 1, bits          # a consumer gave up its wait on a full barrier
        # only wait bits: pipeline waits (1, 2) and, since the item whose stage
        # was skipped never publishes its h, the down items' wait for h (32)
        assert bits & ~(1 | 2 | 32) == 0, bits
        # the hook is one-shot: the next call is clean and correct
        mq.moe_quant_forward(layer.cfg, T, x, layer.router_w, layer.bias, layer.table, layer.fmts, out,
                             workspace=ws, ws_bytes=wsb)
        assert mq.moe_quant_status(layer.cfg, T, ws, wsb) == 0
    finally:
        mq.mq_set_path(0)
    y = out.cpu().numpy()
    ry, _, _ = layer.oracle_forward(orc, x_bits)
    assert_close(y, ry)


def test_forward_zero_tokens_is_noop(torch_cuda):
    import torch
    mq = mq_lib()
    spec = get_config("tiny")
    layer = DeviceLayer(spec, 0)
    out = torch.full((1, spec.hidden), 7.0, device="cuda")
    wsb = mq.moe_quant_workspace_size(layer.cfg, 0)
    ws = torch.empty(max(wsb, 256), dtype=torch.uint8, device="cuda")
    x = torch.zeros((1, spec.hidden), dtype=torch.int16, device="cuda")
    mq.moe_quant_forward(layer.cfg, 0, x, layer.router_w, layer.bias, layer.table, layer.fmts, out,
                         workspace=ws, ws_bytes=wsb)
    torch.cuda.synchronize()
    assert (out == 7.0).all()
