"""Activation edge cases on every expert-FFN path (decode mma.sync GEMV,
decode tcgen05 GEMV, prefill grouped GEMM) against the oracle:

  - an all-zero token (its output must be exactly zero);
  - a token whose every 32-element block mixes magnitudes 1e-4 and 1e4;
  - tokens far beyond the fp16 range (entries around 2^48 ~ 2.8e14; the
    SwiGLU outputs then reach ~2^100), which the prefill path handles with a
    per-token power-of-two scale;
  - ordinary N(0, 1) tokens in the same batch.

Each token is compared with its own scale: max |y_t - ref_t| <= 2e-3 max |ref_t|
(a batch-wide scale would hide the small tokens behind the large ones).
The literal bf16 maximum is not used: with it the layer output itself
overflows fp32 in the oracle, so there is nothing finite to compare."""
from dataclasses import replace

import numpy as np
import pytest

from tests.gpu_helpers import DeviceLayer, assert_close, mq_lib
from workloads.configs import LayerSpec
from workloads.synth import f32_to_bf16_bits, rng_for

pytestmark = pytest.mark.gpu

SMALL = LayerSpec(name="edge_mixed", hidden=512, inter=256, n_experts=12, n_groups=4, topk_group=2, top_k=3,
                  tokens=6, has_shared=True, mixed=True, router_std=1 / 22.6, bias_std=0.01)
FMTS = np.array([[1, 2, 3], [2, 3, 4], [3, 4, 1], [4, 1, 2]] * 3 + [[4, 4, 4]], np.uint8)


@pytest.fixture(scope="module")
def torch_cuda():
    import torch
    assert torch.cuda.is_available()
    return torch


def edge_tokens(H: int, seed: int) -> np.ndarray:
    r = rng_for(seed)
    x = r.standard_normal((6, H), dtype=np.float32)
    x[0] = 0.0                                                          # all zero
    x[1] *= np.where(r.random(H) < 0.5, np.float32(1e-4), np.float32(1e4))   # 1e-4 and 1e4 in every block
    x[2] *= np.float32(2.0 ** 48)                                       # far beyond fp16
    x[3, ::7] *= np.float32(2.0 ** 40)                                  # a few huge entries among N(0, 1)
    return f32_to_bf16_bits(x)


@pytest.mark.parametrize("path", [1, 3, 2], ids=["decode_mma", "decode_tc", "prefill"])
def test_activation_edge_cases(torch_cuda, orc, path):
    mq = mq_lib()
    layer = DeviceLayer(SMALL, 31, fmts=FMTS)
    x = edge_tokens(SMALL.hidden, 77)
    mq.mq_set_path(path)
    try:
        y, idx, w = layer.forward(x)
        status = mq.moe_quant_status(layer.cfg, x.shape[0], *_last_ws(layer, x))
    finally:
        mq.mq_set_path(0)
    assert status == 0
    ry, ridx, rw = layer.oracle_forward(orc, x)
    np.testing.assert_array_equal(idx, ridx)
    np.testing.assert_array_equal(w.view(np.uint32), rw.view(np.uint32))
    assert np.isfinite(ry).all()
    assert (y[0] == 0.0).all() and (ry[0] == 0.0).all()
    for t in range(1, x.shape[0]):
        assert_close(y[t:t + 1], ry[t:t + 1])


def _last_ws(layer, x):
    """A workspace holding the error word of a fresh call with these inputs
    (DeviceLayer.forward allocates its own and drops it)."""
    import torch
    mq = mq_lib()
    T = x.shape[0]
    xd = torch.from_numpy(np.ascontiguousarray(x).view(np.int16)).cuda()
    out = torch.empty((T, layer.spec.hidden), device="cuda")
    wsb = mq.moe_quant_workspace_size(layer.cfg, T)
    ws = torch.empty(wsb, dtype=torch.uint8, device="cuda")
    mq.moe_quant_forward(layer.cfg, T, xd, layer.router_w, layer.bias, layer.table, layer.fmts, out,
                         workspace=ws, ws_bytes=wsb)
    return ws, wsb


@pytest.mark.parametrize("path", [1, 2], ids=["decode_mma", "prefill"])
def test_edge_tokens_on_a_v3_layer(torch_cuda, orc, path):
    """The same edge tokens through a V3-shaped layer (hidden 7168, Q2_K /
    Q3_K / Q8_0), routed against the oracle one call."""
    from workloads import get_config
    spec = replace(get_config("v3_decode_t1"), tokens=6)
    layer = DeviceLayer(spec, 3)
    x = edge_tokens(spec.hidden, 78)
    mq = mq_lib()
    mq.mq_set_path(path)
    try:
        y, idx, w = layer.forward(x)
    finally:
        mq.mq_set_path(0)
    orc.use_openmp(True)
    try:
        ry, ridx, rw = layer.oracle_forward(orc, x, idx_hint=idx)
    finally:
        orc.use_openmp(False)
    np.testing.assert_array_equal(idx, ridx)
    assert (y[0] == 0.0).all()
    for t in range(1, x.shape[0]):
        assert_close(y[t:t + 1], ry[t:t + 1])
