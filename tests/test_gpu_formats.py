"""Q6_K-style and BF16 expert tensors (Sec. 3.3: the planner's upgrade
targets and unquantized tensors) on the GPU: device unpack bit-exact, and
layers mixing them with the other formats through the decode GEMV kernels
and the prefill grouped GEMM, against the oracle."""
from dataclasses import replace

import numpy as np
import pytest

from tests.gpu_helpers import DeviceLayer, assert_close, mq_lib, tokens
from workloads.configs import LayerSpec
from workloads.synth import random_packed, rng_for

pytestmark = pytest.mark.gpu

Q2, Q3, Q4, Q8, Q6, BF = 1, 2, 3, 4, 5, 6


@pytest.fixture(scope="module")
def torch_cuda():
    import torch
    assert torch.cuda.is_available()
    return torch


@pytest.mark.parametrize("fmt", [Q6, BF])
@pytest.mark.parametrize("shape", [(16, 256), (33, 300), (128, 7168), (7168, 2048)])
def test_unpack_device_bit_exact(torch_cuda, orc, fmt, shape):
    mq = mq_lib()
    rows, cols = shape
    p = random_packed(fmt, rows, cols, rng_for(fmt * 131 + rows))
    dev = torch_cuda.from_numpy(p).cuda()
    out = torch_cuda.empty((rows, cols), dtype=torch_cuda.float32, device="cuda")
    mq.mq_unpack_device(fmt, dev, rows, cols, out)
    np.testing.assert_array_equal(out.cpu().numpy().view(np.uint32), orc.unpack(fmt, p, rows, cols).view(np.uint32))


# every expert mixes the new formats with the old; the shared expert is Q6_K / BF16
UPG = LayerSpec(name="upgrade_mixed", hidden=512, inter=256, n_experts=12, n_groups=4, topk_group=2, top_k=3,
                tokens=1, has_shared=True, mixed=True, router_std=1 / 22.6, bias_std=0.01)
UPG_FMTS = np.array([[Q6, Q6, Q6], [BF, BF, BF], [Q6, BF, Q2], [BF, Q6, Q3], [Q2, Q6, BF], [Q8, BF, Q6],
                     [Q4, Q6, Q6], [Q6, Q3, BF], [BF, Q2, Q8], [Q3, BF, Q4], [Q6, Q4, BF], [BF, Q8, Q6],
                     [Q6, BF, Q6]], np.uint8)


@pytest.fixture(params=[1, 2], ids=["decode", "prefill"])
def path(request):
    mq = mq_lib()
    mq.mq_set_path(request.param)
    yield request.param
    mq.mq_set_path(0)


@pytest.mark.parametrize("T", [1, 3, 5, 9, 64, 70])
def test_forward_upgrade_formats(torch_cuda, orc, path, T):
    spec = replace(UPG, tokens=T)
    layer = DeviceLayer(spec, 200 + T, fmts=UPG_FMTS)
    x = tokens(spec, 200 + T)
    y, idx, w = layer.forward(x)
    ry, ridx, rw = layer.oracle_forward(orc, x)
    np.testing.assert_array_equal(idx, ridx)
    np.testing.assert_array_equal(w.view(np.uint32), rw.view(np.uint32))
    assert_close(y, ry)


@pytest.mark.parametrize("T", [1, 4])
def test_forward_v3_shaped_shared_q6k_and_bf16(torch_cuda, orc, T):
    """V3 shapes (hidden 7168, inter 2048, 192 experts, top-8) with the
    shared expert upgraded (gate/up Q6_K, down BF16) and routed experts drawn
    from all six formats, on the decode kernels."""
    mq = mq_lib()
    from workloads import get_config
    spec = replace(get_config("v3_decode_t1"), tokens=T)
    r = rng_for(77 + T)
    fmts = r.choice(np.array([Q2, Q3, Q4, Q8, Q6, BF], np.uint8), size=(spec.n_experts + 1, 3))
    fmts[spec.n_experts] = (Q6, Q6, BF)
    layer = DeviceLayer(spec, 300 + T, fmts=fmts)
    x = tokens(spec, 300 + T)
    mq.mq_set_path(1)
    try:
        y, idx, w = layer.forward(x)
    finally:
        mq.mq_set_path(0)
    ry, ridx, _ = layer.oracle_forward(orc, x, idx_hint=idx)
    np.testing.assert_array_equal(idx, ridx)
    assert_close(y, ry)


def test_tcgen05_gemv_refuses_upgrade_formats_and_auto_goes_to_gemm(torch_cuda, orc):
    """Shapes that are multiples of 128 but not 256 take the tcgen05 GEMV
    kernels at decode; those do not take Q6_K / BF16: a forced request is
    refused (MQ_EFORMAT, nothing enqueued), the automatic choice runs the
    grouped GEMM instead and matches the oracle."""
    mq = mq_lib()
    spec = replace(UPG, hidden=384, inter=128, tokens=2)
    layer = DeviceLayer(spec, 5, fmts=UPG_FMTS)
    x = tokens(spec, 5)
    mq.mq_set_path(3)
    try:
        with pytest.raises(mq.MoeqError) as ei:
            layer.forward(x)
        assert ei.value.status == mq.MQ_EFORMAT
    finally:
        mq.mq_set_path(0)
    y, idx, _ = layer.forward(x)
    ry, ridx, _ = layer.oracle_forward(orc, x)
    np.testing.assert_array_equal(idx, ridx)
    assert_close(y, ry)


def _bf16_big_layer(torch_cuda, big):
    """UPG with expert 1 (all BF16) given one weight of magnitude `big`."""
    spec = replace(UPG, tokens=64)
    layer = DeviceLayer(spec, 9, fmts=UPG_FMTS)
    t = layer.tensors[1][0]                       # expert 1 gate, BF16
    bits = np.array([np.float32(big)]).view(np.uint32)[0] >> 16
    t[0:2] = torch_cuda.from_numpy(np.array([bits & 0xFF, bits >> 8], np.uint8)).cuda()
    return spec, layer


def test_prefill_flags_bf16_weights_beyond_fp16(torch_cuda):
    """A BF16 weight the prefill GEMM's fp16 operands cannot hold sets bit 64
    of the error word (MQ_EDEVICE) instead of passing an infinity on (the
    infinite gate sum then also trips the SwiGLU range check, bit 16); a large
    one that fits sets nothing."""
    mq = mq_lib()
    for big, want in ((2.0 ** 17, 64 | 16), (40000.0, 0)):
        spec, layer = _bf16_big_layer(torch_cuda, big)
        x = torch_cuda.from_numpy(np.ascontiguousarray(tokens(spec, 9)).view(np.int16)).cuda()
        out = torch_cuda.empty((spec.tokens, spec.hidden), dtype=torch_cuda.float32, device="cuda")
        # the 64 tokens must select expert 1 at least once (checked below)
        idx = torch_cuda.empty((spec.tokens, spec.top_k), dtype=torch_cuda.int32, device="cuda")
        wts = torch_cuda.empty((spec.tokens, spec.top_k), dtype=torch_cuda.float32, device="cuda")
        wsb = mq.moe_quant_workspace_size(layer.cfg, spec.tokens)
        ws = torch_cuda.empty(wsb, dtype=torch_cuda.uint8, device="cuda")
        mq.mq_set_path(2)
        try:
            mq.moe_quant_forward(layer.cfg, spec.tokens, x, layer.router_w, layer.bias, layer.table, layer.fmts, out,
                                 idx, wts, ws, wsb)
            bits = mq.moe_quant_status(layer.cfg, spec.tokens, ws, wsb)
        finally:
            mq.mq_set_path(0)
        assert (idx.cpu().numpy() == 1).any()
        assert bits == want, (big, bits)
