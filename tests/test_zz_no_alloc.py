"""moe_quant_forward_noalloc: the forward pass for callers that cannot
allocate device memory (a plugin whose host owns all allocations, serving
loops that must not call cudaMalloc/cudaFree because those can synchronize
the device).  Its scratch is a fixed 16 MiB device array inside the library,
so the test checks that its output is bit-identical to the workspace-based
moe_quant_forward (both run the same deterministic kernels; only the scratch
differs) on two calls in a row (the second call sees the first call's
leftovers in the shared array) and that requests larger than the array are
refused before anything is enqueued.

This file is collected last on purpose, and it must pass both on its own in a
fresh process (the first call on the device does the address lookup) and
after every other test."""
from __future__ import annotations

import numpy as np
import pytest

from workloads.configs import LayerSpec
from tests.gpu_helpers import DeviceLayer, mq_lib, tokens

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def torch_cuda():
    import torch
    assert torch.cuda.is_available()
    return torch


def _run_noalloc(lay: DeviceLayer, x_bits: np.ndarray):
    import torch
    mq = mq_lib()
    T, spec = x_bits.shape[0], lay.spec
    x = torch.from_numpy(np.ascontiguousarray(x_bits).view(np.int16)).cuda()
    out = torch.full((T, spec.hidden), float("nan"), device="cuda")
    idx = torch.full((T, spec.top_k), -1, dtype=torch.int32, device="cuda")
    w = torch.zeros((T, spec.top_k), dtype=torch.float32, device="cuda")
    mq.moe_quant_forward_noalloc(lay.cfg, T, x, lay.router_w, lay.bias, lay.table, lay.fmts, out, idx, w)
    torch.cuda.synchronize()
    return out.cpu().numpy(), idx.cpu().numpy(), w.cpu().numpy()


def test_noalloc_matches_workspace_forward_twice(torch_cuda):
    spec = LayerSpec(name="noalloc", hidden=512, inter=256, n_experts=16, n_groups=4, topk_group=2, top_k=3,
                     tokens=5, has_shared=True, mixed=True, router_std=1 / 22.6, bias_std=0.01)
    lay = DeviceLayer(spec, 23)
    # two different batches: the second call must not depend on what the
    # first one left in the shared scratch
    for call, seed in enumerate((5, 6)):
        x = tokens(spec, seed, 5 + call)
        ref, ridx, rw = lay.forward(x)
        y, idx, w = _run_noalloc(lay, x)
        assert mq_lib().moe_quant_status_noalloc(lay.cfg, x.shape[0]) == 0   # no wait gave up
        np.testing.assert_array_equal(idx, ridx)
        np.testing.assert_array_equal(w, rw)
        assert np.isfinite(y).all()
        np.testing.assert_array_equal(y.view(np.uint32), ref.view(np.uint32))


def test_noalloc_refuses_requests_beyond_its_scratch(torch_cuda):
    mq = mq_lib()
    cfg = mq.make_cfg(7168, 2048, 192, 8, 4, 8, 1.0, True)
    T = 64   # needs about 30 MiB of scratch
    assert mq.moe_quant_workspace_size(cfg, T) > 16 << 20
    table = mq.ExpertTable([(16, 16, 16)] * 192, (16, 16, 16))
    fmts = np.full((193, 3), 1, np.uint8)
    rc = mq._lib.moe_quant_forward_noalloc(mq.ctypes.byref(cfg), T, 16, 16, 16, mq.ctypes.byref(table.table),
                                           fmts.ctypes.data, 16, None, None, None)
    assert rc == mq.MQ_ERANGE
