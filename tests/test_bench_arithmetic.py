"""The numbers the roofline fractions rest on, counted by hand.

bench.py divides algorithmic bytes (decode) or FLOPs (prefill) per launch by
the measured duration.  These tests fix those counts for the V3 workloads
from the format definitions alone (bytes per 256- or 32-weight block), so a
slip in bench.py's accounting (a tensor counted twice, a missing shared
expert, a wrong row count) shows up on the CPU.

Per-block bytes of the formats (planes: fp16 d, fp16 dmin, scale record,
codes, high bits): Q2_K 2 + 2 + 16 + 64 = 84 per 256 weights, Q3_K
2 + 12 + 64 + 32 = 110 per 256, Q8_0 2 + 32 = 34 per 32.  A V3 expert has
gate and up of 2048 x 7168 and down of 7168 x 2048 weights.
"""
from __future__ import annotations

import numpy as np

H, I = 7168, 2048
GATE_Q2K = I * (H // 256) * 84            # 4,816,896 B
DOWN_Q3K = H * (I // 256) * 110           # 6,307,840 B
SHARED_Q80 = 3 * I * (H // 32) * 34       # 46,792,704 B (gate, up and down)


def test_hand_counts_match_the_planar_layout_sizes():
    # every plane of these tensors is a whole number of 256-byte units, so
    # the planar layout adds no padding to the per-block counts
    from workloads.configs import Q2_K, Q3_K, Q8_0, packed_bytes
    assert packed_bytes(Q2_K, I, H) == GATE_Q2K == 4_816_896
    assert packed_bytes(Q3_K, H, I) == DOWN_Q3K == 6_307_840
    assert 2 * packed_bytes(Q8_0, I, H) + packed_bytes(Q8_0, H, I) == SHARED_Q80 == 46_792_704


def test_v3_decode_one_token_algorithmic_bytes():
    import bench
    from workloads.configs import get_config
    from workloads.synth import draw_formats
    spec = get_config("v3_decode_t1")
    fmts = draw_formats(spec, 0)
    idx = np.array([[5, 17, 40, 41, 99, 120, 150, 191]], np.int32)   # eight distinct experts
    b = bench.step_bytes(spec, fmts, [idx])[0]
    quantized = 8 * (2 * GATE_Q2K + DOWN_Q3K) + SHARED_Q80
    assert b["quantized"] == quantized == 174_325_760
    # plus the bf16 token (read by gate/up), the fp32 h of 8 routed + 1
    # shared assignments written by gate/up and read by down, and the fp32
    # output row written by down
    assert b["ffn_mma"] == quantized + H * 2 + 2 * (8 + 1) * I * 4 + H * 4 == 174_516_224


def test_v3_prefill_dense_flops_and_active_flops():
    import bench
    from workloads.configs import get_config
    spec = get_config("v3_prefill_t2048_zipf")
    rows = 2048 * 8 + 2048                 # routed assignments plus the shared expert's rows
    f = bench.step_flops(spec)
    assert f["gateup_tc"] == rows * 2 * (2 * H * I) == 1_082_331_758_592
    assert f["down_tc"] == rows * 2 * H * I
    P = 3 * H * I                           # parameters of one routed expert
    a = bench.flops_active_per_token([8], P, True)
    assert a["routed"] == 2 * 8 * P == 704_643_072
    assert a["with_shared"] == 2 * 9 * P
