"""Helpers for the GPU parity tests: build a layer's inputs on the device
from the seeded generators, run the library through its C ABI, run the
oracle on host copies of the same bytes, and compare."""
from __future__ import annotations

import numpy as np

from workloads.configs import LayerSpec
from workloads.synth import (draw_formats, draw_fp32_weights, draw_router, draw_tokens, random_packed_device,
                             tensor_shapes)

TOL = 2e-3   # max |y_gpu - y_ref| <= TOL * max |y_ref|  (fp32 accumulation)


def mq_lib():
    import paper_2509_25689_gb300 as mq
    return mq


class DeviceLayer:
    """Packed expert tensors of one layer resident on the GPU."""

    def __init__(self, spec: LayerSpec, seed: int, fmts: np.ndarray | None = None, orc=None):
        import torch
        self.spec, self.seed = spec, seed
        self.fmts = draw_formats(spec, seed) if fmts is None else np.asarray(fmts, np.uint8)
        n = spec.n_experts + (1 if spec.has_shared else 0)
        self.tensors = []
        mq = mq_lib()
        if spec.quantize_from_fp32:
            # real fp32 weights packed by the library's host quantizer; the
            # oracle packs the same weights itself and the bytes must agree
            ws = draw_fp32_weights(spec, seed)
            for e in range(n):
                trip = []
                for j in range(3):
                    p = mq.mq_pack(int(self.fmts[e, j]), ws[e][j])
                    if orc is not None:
                        np.testing.assert_array_equal(p, orc.pack(int(self.fmts[e, j]), ws[e][j]))
                    trip.append(torch.from_numpy(p).cuda())
                self.tensors.append(tuple(trip))
        else:
            gen = torch.Generator(device="cuda")
            gen.manual_seed(seed * 7919 + 13)
            shapes = tensor_shapes(spec)
            for e in range(n):
                self.tensors.append(tuple(random_packed_device(int(self.fmts[e, j]), *shapes[j], gen, "cuda")
                                          for j in range(3)))
        routed = self.tensors[:spec.n_experts]
        shared = self.tensors[spec.n_experts] if spec.has_shared else None
        self.table = mq.ExpertTable(routed, shared)
        rw, b = draw_router(spec, seed)
        self.router_w_host, self.bias_host = rw, b
        self.router_w = torch.from_numpy(rw).cuda()
        self.bias = torch.from_numpy(b).cuda()
        self.cfg = mq.make_cfg(spec.hidden, spec.inter, spec.n_experts, spec.n_groups, spec.topk_group,
                               spec.top_k, spec.routed_scale, spec.has_shared)

    def host_tensor(self, e: int, j: int) -> np.ndarray:
        return self.tensors[e][j].cpu().numpy()

    def forward(self, x_bits: np.ndarray):
        import torch
        mq = mq_lib()
        T = x_bits.shape[0]
        spec = self.spec
        x = torch.from_numpy(np.ascontiguousarray(x_bits).view(np.int16)).cuda()
        out = torch.full((T, spec.hidden), float("nan"), device="cuda")
        idx = torch.full((T, spec.top_k), -1, dtype=torch.int32, device="cuda")
        w = torch.zeros((T, spec.top_k), dtype=torch.float32, device="cuda")
        wsb = mq.moe_quant_workspace_size(self.cfg, T)
        ws = torch.empty(wsb, dtype=torch.uint8, device="cuda")
        mq.moe_quant_forward(self.cfg, T, x, self.router_w, self.bias, self.table, self.fmts, out, idx, w, ws, wsb)
        torch.cuda.synchronize()
        return out.cpu().numpy(), idx.cpu().numpy(), w.cpu().numpy()

    def oracle_forward(self, orc, x_bits: np.ndarray, idx_hint: np.ndarray | None = None):
        spec = self.spec
        n = spec.n_experts + (1 if spec.has_shared else 0)
        used = set(range(spec.n_experts, n))
        if idx_hint is not None:
            used |= set(int(e) for e in idx_hint.reshape(-1))
        else:
            used |= set(range(spec.n_experts))
        dummy = np.zeros(16, np.uint8)
        gate, up, down = [], [], []
        for e in range(n):
            if e in used:
                gate.append(self.host_tensor(e, 0)); up.append(self.host_tensor(e, 1)); down.append(self.host_tensor(e, 2))
            else:
                gate.append(dummy); up.append(dummy); down.append(dummy)
        layer = orc.make_layer(spec.hidden, spec.inter, spec.n_experts, spec.n_groups, spec.topk_group, spec.top_k,
                               spec.routed_scale, spec.has_shared)
        return orc.moe_forward(layer, x_bits, self.router_w_host, self.bias_host, gate, up, down, self.fmts)


def assert_close(y, ref, tol=TOL):
    scale = float(np.abs(ref).max())
    err = float(np.abs(y.astype(np.float64) - ref.astype(np.float64)).max())
    assert np.isfinite(y).all()
    assert err <= tol * scale, f"max err {err:.3e} > {tol} * {scale:.3e}"
    return err / max(scale, 1e-30)


def tokens(spec: LayerSpec, seed: int, T: int | None = None) -> np.ndarray:
    return draw_tokens(seed + 101, spec.tokens if T is None else T, spec.hidden)
