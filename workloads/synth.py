"""Seeded input generators (numpy PCG64 on the host, torch's generator on a
CUDA device).  Nothing here quantizes, dequantizes or routes: packed tensors
for the V3-shaped layers are drawn directly as random plane contents (any
code / scale byte is a valid field; the fp16 scale planes get positive
values in a range that makes the decoded weights look like N(0, 0.02)), and
the tiny layer's fp32 weights are returned unpacked for a packer to consume.

Recipe (stated here and in the design notes):
  x           bf16 ~ N(0, 1)           (fp32 draw rounded to nearest-even bf16)
  router_w    fp32 ~ N(0, router_std)  (1/sqrt(hidden))
  bias        fp32 ~ N(0, bias_std)    (0.01 on V3 layers, 0 on the tiny layer)
  codes/fields uniform random bytes
  d, dmin     fp16 = base * U(0.5, 1.5), base per format (FP16_BASE)
  bf16 tensor bf16 ~ N(0, 0.02)        (BF16 format: values, not fields)
  pruned set  sorted draw of n_experts of the original 256 ids
"""
from __future__ import annotations

import numpy as np

from .configs import PLANES, PLANE_ALIGN, Q2_K, Q3_K, Q4_K, Q6_K, Q8_0, ROW_TILE, LayerSpec, packed_bytes

# fp16 scale bases: decoded weights then have mean ~0 and std ~0.02
FP16_BASE = {
    Q2_K: (1.44e-3, 2.16e-3),
    Q3_K: (4.7e-4,),
    Q4_K: (7.7e-5, 5.8e-4),
    Q8_0: (2.7e-4,),
    Q6_K: (6.5e-5,),      # d straddles the smallest normal fp16 (6.1e-5): both kinds occur
}
BF16_STD = 0.02


def rng_for(seed: int) -> np.random.Generator:
    return np.random.Generator(np.random.PCG64(seed))


def f32_to_bf16_bits(a: np.ndarray) -> np.ndarray:
    u = np.ascontiguousarray(a, dtype=np.float32).view(np.uint32).astype(np.uint64)
    u = (u + 0x7FFF + ((u >> 16) & 1)) >> 16
    return u.astype(np.uint16)


def bf16_bits_to_f32(b: np.ndarray) -> np.ndarray:
    return (np.asarray(b, dtype=np.uint16).astype(np.uint32) << 16).view(np.float32)


def draw_tokens(seed: int, tokens: int, hidden: int) -> np.ndarray:
    """bf16 bits [tokens, hidden] of N(0,1) activations."""
    return f32_to_bf16_bits(rng_for(seed).standard_normal((tokens, hidden), dtype=np.float32))


def draw_formats(spec: LayerSpec, seed: int) -> np.ndarray:
    """uint8 [(E + shared), 3] formats in the order gate, up, down."""
    n = spec.n_experts + (1 if spec.has_shared else 0)
    f = np.zeros((n, 3), np.uint8)
    if spec.mixed:
        r = rng_for(seed + 7)
        vals = np.array([p[0] for p in spec.mixed_probs], np.uint8)
        probs = np.array([p[1] for p in spec.mixed_probs])
        f[: spec.n_experts] = r.choice(vals, size=(spec.n_experts, 3), p=probs)
    else:
        f[: spec.n_experts] = (spec.gate_fmt, spec.up_fmt, spec.down_fmt)
    if spec.has_shared:
        f[spec.n_experts] = spec.shared_fmt
    return f


def zipf_ranks(spec: LayerSpec, seed: int) -> np.ndarray:
    """Seeded popularity rank of every expert (0 = most popular)."""
    return rng_for(seed + 5).permutation(spec.n_experts).astype(np.int64)


def zipf_bias() -> np.ndarray:
    """Per-expert selection bias of the Zipf-skewed prefill workload, fitted
    once through oracle routing (tests/golden/fit_zipf_bias.py) so that the
    routed counts follow the water-filled Zipf(s) target; stored bit-exact."""
    import json
    import os
    path = os.path.join(os.path.dirname(os.path.dirname(os.path.abspath(__file__))), "tests", "golden",
                        "zipf_bias.json")
    with open(path) as f:
        return np.array([float.fromhex(v) for v in json.load(f)["bias_f32_hex"]], np.float32)


def draw_router(spec: LayerSpec, seed: int, base_only: bool = False):
    """Router weights and selection bias.  Zipf-skewed workloads (zipf_s set)
    take the fitted bias instead of the N(0, bias_std) draw unless base_only."""
    r = rng_for(seed + 1)
    w = (r.standard_normal((spec.n_experts, spec.hidden), dtype=np.float32)
         * np.float32(spec.router_std)).astype(np.float32)
    if spec.bias_std > 0:
        b = (r.standard_normal(spec.n_experts, dtype=np.float32) * np.float32(spec.bias_std)).astype(np.float32)
    else:
        b = np.zeros(spec.n_experts, np.float32)
    if spec.zipf_s is not None and not base_only:
        b = zipf_bias()
    return w, b


def pruned_subset(spec: LayerSpec, seed: int) -> np.ndarray:
    """Original expert ids kept by pruning, ascending; index = pruned id."""
    return np.sort(rng_for(seed + 3).choice(spec.n_original_experts, spec.n_experts, replace=False)).astype(np.int32)


def draw_fp32_weights(spec: LayerSpec, seed: int):
    """Tiny layer: fp32 N(0, weight_std) gate/up [I,H] and down [H,I] per expert."""
    r = rng_for(seed + 11)
    n = spec.n_experts + (1 if spec.has_shared else 0)
    out = []
    for _ in range(n):
        g = (r.standard_normal((spec.inter, spec.hidden), dtype=np.float32) * np.float32(spec.weight_std))
        u = (r.standard_normal((spec.inter, spec.hidden), dtype=np.float32) * np.float32(spec.weight_std))
        d = (r.standard_normal((spec.hidden, spec.inter), dtype=np.float32) * np.float32(spec.weight_std))
        out.append((g.astype(np.float32), u.astype(np.float32), d.astype(np.float32)))
    return out


def _plane_layout(fmt: int, rows: int, cols: int):
    qk, planes = PLANES[fmt]
    nblk = (-(-rows // ROW_TILE) * ROW_TILE) * ((cols + qk - 1) // qk)
    off = 0
    out = []
    for kind, b in planes:
        out.append((kind, off, nblk * b))
        off += -(-nblk * b // PLANE_ALIGN) * PLANE_ALIGN
    return nblk, out


def random_packed(fmt: int, rows: int, cols: int, r: np.random.Generator) -> np.ndarray:
    """Random plane contents for a rows x cols tensor in format fmt (host)."""
    nblk, planes = _plane_layout(fmt, rows, cols)
    buf = np.zeros(packed_bytes(fmt, rows, cols), np.uint8)
    fi = 0
    for kind, off, n in planes:
        if kind == "f16":
            base = FP16_BASE[fmt][fi]
            fi += 1
            v = (base * (0.5 + r.random(nblk, dtype=np.float32))).astype(np.float16)
            buf[off:off + n] = v.view(np.uint8)
        elif kind == "bf16":
            v = f32_to_bf16_bits(r.standard_normal(n // 2, dtype=np.float32) * np.float32(BF16_STD))
            buf[off:off + n] = v.view(np.uint8)
        else:
            buf[off:off + n] = np.frombuffer(r.bytes(n), np.uint8)
    return buf


def random_packed_device(fmt: int, rows: int, cols: int, gen, device):
    """Same recipe as random_packed, drawn on a CUDA device with torch's
    generator (plumbing only).  Returns a uint8 device tensor."""
    import torch
    nblk, planes = _plane_layout(fmt, rows, cols)
    buf = torch.zeros(packed_bytes(fmt, rows, cols), dtype=torch.uint8, device=device)
    fi = 0
    for kind, off, n in planes:
        if kind == "f16":
            base = FP16_BASE[fmt][fi]
            fi += 1
            v = (base * (0.5 + torch.rand(nblk, generator=gen, device=device))).to(torch.float16)
            buf[off:off + n] = v.view(torch.uint8)
        elif kind == "bf16":
            v = (torch.randn(n // 2, generator=gen, device=device) * BF16_STD).to(torch.bfloat16)
            buf[off:off + n] = v.view(torch.uint8)
        else:
            buf[off:off + n] = torch.randint(0, 256, (n,), generator=gen, device=device,
                                             dtype=torch.int16).to(torch.uint8)
    return buf


def tensor_shapes(spec: LayerSpec):
    """(rows, cols) of gate, up, down."""
    return (spec.inter, spec.hidden), (spec.inter, spec.hidden), (spec.hidden, spec.inter)


def draw_packed_layer_host(spec: LayerSpec, seed: int, fmts: np.ndarray, experts=None):
    """Host random packed tensors for the listed experts (default: all)."""
    n = spec.n_experts + (1 if spec.has_shared else 0)
    experts = range(n) if experts is None else experts
    shapes = tensor_shapes(spec)
    out = {}
    for e in experts:
        r = rng_for(seed * 100003 + 17 + e)
        out[e] = tuple(random_packed(int(fmts[e, j]), *shapes[j], r) for j in range(3))
    return out


def zipf_target_counts(n_experts: int, total: int, s: float, cap: int) -> np.ndarray:
    """Zipf(s) shares of `total` assignments over ranks, water-filled under a
    per-expert cap (one token picks an expert at most once)."""
    p = (np.arange(1, n_experts + 1, dtype=np.float64)) ** (-s)
    p /= p.sum()
    counts = np.zeros(n_experts)
    free = np.ones(n_experts, bool)
    remaining = float(total)
    for _ in range(n_experts):
        share = p * free
        share = share / share.sum() * remaining
        over = free & (share > cap)
        if not over.any():
            counts[free] = share[free]
            break
        counts[over] = cap
        remaining -= cap * over.sum()
        free &= ~over
    return counts
