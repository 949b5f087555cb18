"""CPU tests of the C ABI: the library loads and exports every symbol that
include/moeq.h declares, the host codec is byte-identical to the oracle's
quantizer/dequantizer, and argument checks reject bad calls before any GPU
work (no GPU needed for any of these)."""
import ctypes
import os
import re

import numpy as np
import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def mq():
    import __graft_entry__
    __graft_entry__.build()
    import paper_2509_25689_gb300 as m
    return m


def _declared_functions():
    import glob
    src = ""
    for h in sorted(glob.glob(os.path.join(ROOT, "include", "*.h"))):
        with open(h) as f:
            src += f.read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    names = re.findall(r"^\s*(?:const\s+)?[A-Za-z_][A-Za-z0-9_]*\s*\*?\s*([a-z_][a-z0-9_]*)\s*\(", src, flags=re.M)
    return sorted(set(n for n in names if n.startswith(("mq_", "moe_"))))


def test_library_exports_every_declared_symbol(mq):
    names = _declared_functions()
    assert len(names) >= 14
    lib = ctypes.CDLL(mq.LIB_PATH)
    for n in names:
        assert hasattr(lib, n), n
        assert n in mq.EXPORTED, n


@pytest.mark.parametrize("fmt", ["Q2_K", "Q3_K", "Q4_K", "Q8_0", "Q6_K", "BF16"])
@pytest.mark.parametrize("shape", [(1, 32), (3, 256), (5, 300), (16, 1024), (7, 2051)])
def test_host_pack_unpack_match_oracle(mq, orc, fmt, shape):
    rng = np.random.default_rng(hash((fmt, shape)) % 2**32)
    w = rng.normal(0, 0.02, shape).astype(np.float32)
    w[:, :3] *= 40.0   # a few outliers per row
    a, b = mq.mq_pack(fmt, w), orc.pack(fmt, w)
    np.testing.assert_array_equal(a, b)
    np.testing.assert_array_equal(mq.mq_unpack(fmt, a, *shape), orc.unpack(fmt, b, *shape))
    assert mq.mq_packed_size(fmt, *shape) == orc.packed_size(fmt, *shape)


@pytest.mark.parametrize("fmt", [1, 2, 3, 4, 5, 6])
def test_host_unpack_random_planes_match_oracle(mq, orc, fmt):
    from workloads.synth import random_packed, rng_for
    p = random_packed(fmt, 9, 768, rng_for(fmt))
    np.testing.assert_array_equal(mq.mq_unpack(fmt, p, 9, 768), orc.unpack(fmt, p, 9, 768))


def test_bad_format_and_sizes(mq):
    assert mq.mq_packed_size(7, 4, 256) == 0
    assert mq.mq_packed_size(1, -1, 256) == 0
    with pytest.raises(mq.MoeqError):
        mq.mq_pack(9, np.zeros((1, 32), np.float32))
    with pytest.raises(mq.MoeqError):
        mq.mq_pack("Q8_0", np.full((1, 32), np.inf, np.float32))
    with pytest.raises(mq.MoeqError):       # rounds past the largest bf16
        mq.mq_pack("BF16", np.full((1, 32), np.finfo(np.float32).max, np.float32))


@pytest.mark.parametrize("field,value,code", [
    ("hidden", 100, -4), ("inter", 0, -4), ("n_experts", 300, -4), ("n_groups", 5, -4),
    ("topk_group", 9, -4), ("top_k", 33, -4), ("top_k", 0, -4),
])
def test_shape_checks_reject_before_launch(mq, field, value, code):
    cfg = mq.make_cfg(7168, 2048, 192, 8, 4, 8, has_shared=True)
    setattr(cfg, field, value)
    assert mq.moe_quant_workspace_size(cfg, 1) == 0
    table = mq.ExpertTable([(16, 16, 16)] * 192, shared=(16, 16, 16))
    rc = mq._lib.moe_quant_forward(ctypes.byref(cfg), 1, 16, 16, None, ctypes.byref(table.table),
                                   np.full(193 * 3, 1, np.uint8).ctypes.data, 16, None, None, 256, 1 << 30, None)
    assert rc == code


def test_topk_exceeding_kept_groups_is_rejected(mq):
    cfg = mq.make_cfg(7168, 2048, 192, 8, 1, 25)   # 1 group of 24 cannot supply 25
    assert mq.moe_quant_workspace_size(cfg, 1) == 0


def test_pointer_and_workspace_checks(mq):
    cfg = mq.make_cfg(256, 128, 8, 1, 1, 2)
    ws = mq.moe_quant_workspace_size(cfg, 4)
    assert ws > 0 and ws % 256 == 0
    fmt = np.full(24, 3, np.uint8)
    ok = mq.ExpertTable([(256, 256, 256)] * 8)
    f = lambda x=256, rw=256, table=ok, fm=fmt, out=256, wsp=256, wsb=ws: mq._lib.moe_quant_forward(
        ctypes.byref(cfg), 4, x, rw, None, ctypes.byref(table.table), fm.ctypes.data, out, None, None, wsp, wsb, None)
    assert f(x=0) == -1                         # null activations
    assert f(x=8) == -3                         # misaligned activations
    assert f(wsb=ws - 1) == -5                  # workspace too small
    assert f(wsp=128) == -5                     # workspace not 256-byte aligned
    assert f(table=mq.ExpertTable([(256, 256, 8)] * 8)) == -3   # misaligned packed tensor
    assert f(table=mq.ExpertTable([(256, 0, 256)] * 8)) == -1   # null packed tensor
    bad = fmt.copy(); bad[5] = 9
    assert f(fm=bad) == -2                      # unknown format
    cfg.has_shared = 1
    assert f(wsb=mq.moe_quant_workspace_size(cfg, 4)) == -1     # shared expert missing


def test_strerror(mq):
    assert mq.mq_strerror(0) == "ok"
    assert "workspace" in mq.mq_strerror(-5)


@pytest.mark.parametrize("fmt", [1, 2, 3, 4, 5, 6])
def test_generator_sizes_match_library_and_oracle(mq, orc, fmt):
    # the input generators and bench.py's byte accounting size packed tensors
    # themselves; they must agree with both codecs
    from workloads.configs import packed_bytes
    for rows, cols in [(1, 32), (31, 256), (33, 257), (128, 2048), (2048, 7168), (7168, 2048), (96, 8192)]:
        n = packed_bytes(fmt, rows, cols)
        assert n == mq.mq_packed_size(fmt, rows, cols) == orc.packed_size(fmt, rows, cols), (rows, cols)


def test_bench_step_bytes_counts_each_touched_expert_once(mq):
    import bench
    from workloads.configs import get_config
    spec = get_config("v3_decode_t1")
    E, H, I, K = spec.n_experts, spec.hidden, spec.inter, spec.top_k
    fmts = np.tile(np.array([[1, 1, 2]], np.uint8), (E + 1, 1))
    fmts[E] = 4
    idx = np.array([[3, 7, 7, 11, 0, 190, 191, 3]], np.int32)   # 6 distinct experts
    b = bench.step_bytes(spec, fmts, [idx])[0]
    gu = 2 * mq.mq_packed_size(1, I, H)
    dn = mq.mq_packed_size(2, H, I)
    sh = 2 * mq.mq_packed_size(4, I, H) + mq.mq_packed_size(4, H, I)
    assert b["quantized"] == 6 * (gu + dn) + sh
    assert b["gateup_mma"] == 6 * gu + 2 * mq.mq_packed_size(4, I, H) + H * 2 + (K + 1) * I * 4
    assert b["down_mma"] == 6 * dn + mq.mq_packed_size(4, H, I) + (K + 1) * I * 4 + H * 4
    assert b["ffn_mma"] == b["gateup_mma"] + b["down_mma"]   # the one decode FFN kernel reads both
    assert b["router_logits"] == E * H * 4 + H * 2 + E * 4


def test_binding_refuses_short_buffers(mq):
    w = np.zeros((4, 256), np.float32)
    n = mq.mq_packed_size("Q4_K", 4, 256)
    with pytest.raises(mq.MoeqError):
        mq.mq_pack("Q4_K", w, dst=np.empty(n - 1, np.uint8))
    p = mq.mq_pack("Q4_K", w)
    with pytest.raises(mq.MoeqError):
        mq.mq_unpack("Q4_K", p[: n - 16], 4, 256)
    np.testing.assert_array_equal(mq.mq_unpack("Q4_K", p, 4, 256), w)


def test_bench_traffic_only_for_the_captured_workload():
    import bench
    t = bench._profiled_traffic("ffn_mma")
    assert t is None or t > 0
    assert bench._profiled_traffic("ffn_mma", "v3_decode_t1_k6") is None
    assert bench._profiled_traffic("router_logits") is None


def test_status_argument_checks(mq):
    cfg = mq.make_cfg(256, 128, 8, 1, 1, 2)
    ws = mq.moe_quant_workspace_size(cfg, 4)
    with pytest.raises(mq.MoeqError) as e:
        mq.moe_quant_status(cfg, 4, None, ws)
    assert e.value.status == mq.MQ_EWORKSPACE
    with pytest.raises(mq.MoeqError):
        mq.moe_quant_status(cfg, 4, 256, ws - 1)        # smaller than the forward call's layout
    with pytest.raises(mq.MoeqError):
        mq.moe_quant_status(cfg, 4, 128, ws)            # not 256-byte aligned
    with pytest.raises(mq.MoeqError):
        mq.moe_quant_status(mq.make_cfg(100, 128, 8, 1, 1, 2), 4, 256, ws)
    assert mq.moe_quant_status(cfg, 0, 256, ws) == 0    # no tokens: nothing ran, no device access
    with pytest.raises(mq.MoeqError) as e:
        mq.moe_quant_status_noalloc(mq.make_cfg(7168, 2048, 192, 8, 4, 8, has_shared=True), 4096)
    assert e.value.status == mq.MQ_ERANGE


def test_wait_test_hook_argument_checks(mq):
    for bad in (0, 2_000_000_000):
        with pytest.raises(mq.MoeqError) as e:
            mq.mq_test_fail_next_decode(bad)
        assert e.value.status == mq.MQ_EINVAL
