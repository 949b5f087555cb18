"""Workload definitions: the five synthetic MoE-layer configurations.

Shapes follow the DeepSeek-V3 MoE layer the paper compresses (Sec. 4.1:
256 routed experts pruned with r = 0.75 to 192, shared expert, hidden 7168,
expert intermediate 2048) and a tiny correctness layer.
"""
from __future__ import annotations

import math
from dataclasses import dataclass, field

Q2_K, Q3_K, Q4_K, Q8_0, Q6_K, BF16 = 1, 2, 3, 4, 5, 6
FMT_NAMES = {Q2_K: "Q2_K", Q3_K: "Q3_K", Q4_K: "Q4_K", Q8_0: "Q8_0", Q6_K: "Q6_K", BF16: "BF16"}

# bytes per block in each plane, and weights per block (format geometry used
# only for byte accounting and for filling planes with random content)
PLANES = {
    Q4_K: (256, [("f16", 2), ("f16", 2), ("u8", 12), ("u8", 128)]),
    Q2_K: (256, [("f16", 2), ("f16", 2), ("u8", 16), ("u8", 64)]),
    Q3_K: (256, [("f16", 2), ("u8", 12), ("u8", 64), ("u8", 32)]),
    Q8_0: (32, [("f16", 2), ("u8", 32)]),
    Q6_K: (256, [("f16", 2), ("u8", 16), ("u8", 128), ("u8", 64)]),
    BF16: (32, [("bf16", 64)]),
}
PLANE_ALIGN = 256


ROW_TILE = 32


def packed_bytes(fmt: int, rows: int, cols: int) -> int:
    qk, planes = PLANES[fmt]
    nblk = (-(-rows // ROW_TILE) * ROW_TILE) * ((cols + qk - 1) // qk)
    return sum(-(-nblk * b // PLANE_ALIGN) * PLANE_ALIGN for _, b in planes)


@dataclass
class LayerSpec:
    name: str
    hidden: int
    inter: int
    n_experts: int
    n_groups: int
    topk_group: int
    top_k: int
    tokens: int
    routed_scale: float = 1.0
    has_shared: bool = True
    # per-tensor formats: "fixed" (gate/up/down lists) or "mixed" (drawn)
    gate_fmt: int = Q2_K
    up_fmt: int = Q2_K
    down_fmt: int = Q3_K
    shared_fmt: int = Q8_0
    mixed: bool = False
    mixed_probs: tuple = ((Q2_K, 0.5), (Q3_K, 0.3), (Q4_K, 0.2))
    router_std: float = 0.0
    bias_std: float = 0.0
    weight_std: float = 0.02
    quantize_from_fp32: bool = False   # tiny config: real N(0,0.02) weights packed
    n_original_experts: int = 256
    zipf_s: float | None = None
    n_layers: int = 1
    steps: int = 1
    seed: int = 0
    extra: dict = field(default_factory=dict)

    def expert_param_count(self) -> int:
        return 3 * self.hidden * self.inter


def _v3(**kw) -> LayerSpec:
    base = dict(hidden=7168, inter=2048, n_experts=192, n_groups=8, topk_group=4, top_k=8,
                router_std=1.0 / math.sqrt(7168), bias_std=0.01, has_shared=True)
    base.update(kw)
    return LayerSpec(**base)


CONFIGS = {
    # 1: tiny correctness layer, Q4_K-style, top-2, no groups, 4 tokens
    "tiny": LayerSpec(name="tiny", hidden=256, inter=128, n_experts=8, n_groups=1, topk_group=1,
                      top_k=2, tokens=4, has_shared=False, gate_fmt=Q4_K, up_fmt=Q4_K,
                      down_fmt=Q4_K, router_std=1.0 / 16.0, bias_std=0.0,
                      quantize_from_fp32=True, n_original_experts=8),
    # 2: one V3-shaped layer at decode, 1 token
    "v3_decode_t1": _v3(name="v3_decode_t1", tokens=1),
    # 2 with the paper's deployed activation adjustment: k = ceil(r k_orig) =
    # ceil(0.75 * 8) = 6 experts per token of the 192 kept (Sec. 3.2)
    "v3_decode_t1_k6": _v3(name="v3_decode_t1_k6", tokens=1, top_k=6),
    # 3: 32 decode tokens, per-tensor formats drawn 50/30/20 from Q2_K/Q3_K/Q4_K
    "v3_decode_t32_mixed": _v3(name="v3_decode_t32_mixed", tokens=32, mixed=True),
    # 4: prefill 2048 tokens, Zipf(1.1)-skewed expert counts, mixed formats
    "v3_prefill_t2048_zipf": _v3(name="v3_prefill_t2048_zipf", tokens=2048, mixed=True,
                                 zipf_s=1.1),
    # 5: 20 independent layers, decode at batch 1 and 8, 64 steps
    "v3_stack20": _v3(name="v3_stack20", tokens=1, mixed=True, n_layers=20, steps=64,
                      extra={"batches": (1, 8)}),
    # 5 with per-layer activated experts (Sec. 3.2): k_pruned = ceil(0.75 * 8)
    # = 6, then k_i <= 6 tuned to a budget of 110 expert activations per token
    # over the 20 layers (FLOPs_active = 2 * 110 * P), 10 layers at 5 and 10 at 6
    "v3_stack20_ki": _v3(name="v3_stack20_ki", tokens=1, mixed=True, n_layers=20, steps=64, top_k=6,
                         extra={"batches": (1, 8), "k_orig": 8, "retain": 0.75, "budget_expert_acts": 110}),
}


def get_config(name: str) -> LayerSpec:
    return CONFIGS[name]
