"""Parity of the prefill path (grouped GEMM on the tcgen05 tensor cores, fp16
operands, fp32 accumulation) against the oracle.  The path is forced with
mq_set_path(2) so small layers exercise it too; shapes cover several 128-row
weight tiles, token counts that are not multiples of 16, experts with more
than 256 tokens (several token tiles), every format, and the V3 layer."""
import numpy as np
import pytest

from tests.gpu_helpers import DeviceLayer, assert_close, mq_lib, tokens
from workloads import get_config
from workloads.configs import LayerSpec

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def torch_cuda():
    import torch
    assert torch.cuda.is_available()
    return torch


@pytest.fixture()
def prefill_path():
    mq = mq_lib()
    mq.mq_set_path(2)
    yield
    mq.mq_set_path(0)


def test_prefill_tiny_layer(torch_cuda, orc, prefill_path):
    spec = get_config("tiny")
    layer = DeviceLayer(spec, 0, orc=orc)
    x = tokens(spec, 0)
    y, idx, w = layer.forward(x)
    ry, ridx, rw = layer.oracle_forward(orc, x)
    np.testing.assert_array_equal(idx, ridx)
    assert_close(y, ry)


@pytest.mark.parametrize("T", [1, 5, 17, 40])
def test_prefill_small_mixed_layer_with_shared(torch_cuda, orc, prefill_path, T):
    spec = LayerSpec(name="small_mixed", hidden=512, inter=256, n_experts=12, n_groups=4, topk_group=2,
                     top_k=3, tokens=T, has_shared=True, mixed=True, router_std=1 / 22.6, bias_std=0.01)
    fm = np.array([[1, 2, 3], [2, 3, 4], [3, 4, 1], [4, 1, 2]] * 3 + [[4, 4, 4]], np.uint8)
    layer = DeviceLayer(spec, T, fmts=fm)
    x = tokens(spec, T)
    y, idx, w = layer.forward(x)
    ry, ridx, rw = layer.oracle_forward(orc, x)
    np.testing.assert_array_equal(idx, ridx)
    assert_close(y, ry)


def test_prefill_experts_over_256_tokens(torch_cuda, orc, prefill_path):
    # 4 experts, top-2 of 600 tokens: about 300 tokens per expert and 600 on
    # the shared expert, so units span two or three token tiles
    T = 600
    spec = LayerSpec(name="wide", hidden=384, inter=256, n_experts=4, n_groups=1, topk_group=1, top_k=2,
                     tokens=T, has_shared=True, mixed=True, router_std=1 / 19.6, bias_std=0.0)
    fm = np.array([[1, 2, 3], [3, 1, 2], [2, 3, 4], [4, 4, 1], [3, 4, 2]], np.uint8)
    layer = DeviceLayer(spec, 3, fmts=fm)
    x = tokens(spec, 3, T)
    y, idx, w = layer.forward(x)
    counts = np.bincount(idx.reshape(-1), minlength=4)
    assert counts.max() > 256
    ry, ridx, rw = layer.oracle_forward(orc, x)
    np.testing.assert_array_equal(idx, ridx)
    assert_close(y, ry)


def test_prefill_v3_layer_sampled(torch_cuda, orc, prefill_path):
    spec = get_config("v3_decode_t1")
    layer = DeviceLayer(spec, 0)
    T = 80
    x = tokens(spec, 5, T)
    y, idx, w = layer.forward(x)
    for t in (0, 47, 79):
        ry, ridx, rw = layer.oracle_forward(orc, x[t:t + 1], idx_hint=idx[t])
        np.testing.assert_array_equal(idx[t:t + 1], ridx)
        assert_close(y[t:t + 1], ry)


def _stratified_tokens(idx: np.ndarray, n_experts: int, tile: int = 256, cap: int = 96) -> list:
    """Tokens that exercise the grouped GEMM's corner cases: three on each of
    the hottest expert's second and third token tiles, and the last token of
    every expert's last (partial) tile, thinned evenly to `cap`; padded with
    evenly spaced tokens to at least 64."""
    T = idx.shape[0]
    per_e = [np.nonzero((idx == e).any(axis=1))[0] for e in range(n_experts)]   # ascending = unit order
    hot = int(np.argmax([len(p) for p in per_e]))
    hot_pick = []
    for j in (1, 2):
        tl = per_e[hot][tile * j: tile * (j + 1)]
        if len(tl):
            hot_pick += [int(tl[0]), int(tl[len(tl) // 2]), int(tl[-1])]
    last = sorted({int(p[-1]) for p in per_e if len(p)} - set(hot_pick))
    room = max(0, cap - len(hot_pick))
    if len(last) > room:
        last = [last[i] for i in np.linspace(0, len(last) - 1, room).astype(int)]
    pick = set(hot_pick) | set(last)
    for v in np.linspace(0, T - 1, 64).astype(int):
        if len(pick) >= 64:
            break
        pick.add(int(v))
    return sorted(pick)


def test_prefill_v3_zipf_t2048_stratified(torch_cuda, orc):
    """The Zipf-skewed V3 prefill workload (T = 2048, mixed formats) through
    the automatic path choice, against one oracle call on a stratified sample
    of at least 64 tokens: tokens on the hottest expert's second and third
    256-token tiles, on every expert's last partial tile, and so on every
    format in the layer."""
    spec = get_config("v3_prefill_t2048_zipf")
    layer = DeviceLayer(spec, 0)
    x = tokens(spec, 0)
    y, idx, w = layer.forward(x)
    counts = np.bincount(idx.reshape(-1), minlength=spec.n_experts)
    assert counts.max() >= 4 * counts[counts > 0].mean()   # skewed towards a few experts
    pick = _stratified_tokens(idx, spec.n_experts)
    assert len(pick) >= 64
    used = set(int(e) for e in idx[pick].reshape(-1))
    assert {int(f) for e in used for f in layer.fmts[e]} == {1, 2, 3}   # every routed format
    orc.use_openmp(True)
    try:
        ry, ridx, rw = layer.oracle_forward(orc, x[pick], idx_hint=idx[pick])
    finally:
        orc.use_openmp(False)
    np.testing.assert_array_equal(idx[pick], ridx)
    np.testing.assert_array_equal(w[pick].view(np.uint32), rw.view(np.uint32))
    for i, t in enumerate(pick):
        assert_close(y[t:t + 1], ry[i:i + 1])
