"""Python binding of libmoeq (quantized MoE expert-FFN layer for GB300).

Argument marshalling only: every function forwards to the C ABI entry point
of the same name in libmoeq.so (include/moeq.h).  Tensors may be torch
tensors (device or host) or numpy arrays (host); their data pointers are
passed through.  Importing this module fails loudly if the CUDA library has
not been built: there is no CPU fallback.
"""
from __future__ import annotations

import ctypes
import os

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "libmoeq.so")

MQ_Q2_K, MQ_Q3_K, MQ_Q4_K, MQ_Q8_0, MQ_Q6_K, MQ_BF16 = 1, 2, 3, 4, 5, 6
FORMATS = {"Q2_K": MQ_Q2_K, "Q3_K": MQ_Q3_K, "Q4_K": MQ_Q4_K, "Q8_0": MQ_Q8_0, "Q6_K": MQ_Q6_K, "BF16": MQ_BF16}
MQ_OK = 0
MQ_EINVAL, MQ_EFORMAT, MQ_EALIGN, MQ_ESHAPE, MQ_EWORKSPACE, MQ_ECUDA, MQ_EDEVICE, MQ_ERANGE = range(-1, -9, -1)


class MoeqError(RuntimeError):
    def __init__(self, fn: str, status: int):
        super().__init__(f"{fn}: {mq_strerror(status)} ({status})")
        self.status = status


class mq_layer_cfg(ctypes.Structure):
    _fields_ = [
        ("hidden", ctypes.c_int32), ("inter", ctypes.c_int32), ("n_experts", ctypes.c_int32),
        ("n_groups", ctypes.c_int32), ("topk_group", ctypes.c_int32), ("top_k", ctypes.c_int32),
        ("routed_scale", ctypes.c_float), ("has_shared", ctypes.c_int32),
    ]


class mq_expert_weights(ctypes.Structure):
    _fields_ = [("gate", ctypes.c_void_p), ("up", ctypes.c_void_p), ("down", ctypes.c_void_p)]


class mq_expert_table(ctypes.Structure):
    _fields_ = [("experts", ctypes.POINTER(mq_expert_weights)),
                ("shared", ctypes.POINTER(mq_expert_weights))]


class mq_plan_tensor(ctypes.Structure):
    _fields_ = [("params", ctypes.c_int64), ("layer", ctypes.c_int32), ("kind", ctypes.c_int32),
                ("sens", ctypes.c_double)]


class mq_plan_cfg(ctypes.Structure):
    _fields_ = [("n_levels", ctypes.c_int32), ("bits64", ctypes.POINTER(ctypes.c_int32)),
                ("low", ctypes.c_int32), ("lowest", ctypes.c_int32), ("small_level", ctypes.c_int32),
                ("medium_level", ctypes.c_int32), ("floor_level", ctypes.c_int32),
                ("small_max", ctypes.c_int64), ("medium_max", ctypes.c_int64), ("mem_limit_bytes", ctypes.c_int64)]


class mq_kernel_stat(ctypes.Structure):
    _fields_ = [("name", ctypes.c_char * 48), ("launches", ctypes.c_int32), ("total_ms", ctypes.c_double)]


def _load():
    if not os.path.exists(LIB_PATH):
        raise ImportError(f"libmoeq.so not built ({LIB_PATH}); run paper_2509_25689_gb300/build.py")
    L = ctypes.CDLL(LIB_PATH)
    vp, i32, i64, sz = ctypes.c_void_p, ctypes.c_int32, ctypes.c_int64, ctypes.c_size_t
    cfgp = ctypes.POINTER(mq_layer_cfg)
    sig = {
        "mq_packed_size": (sz, [ctypes.c_int, i64, i64]),
        "mq_pack": (ctypes.c_int, [ctypes.c_int, vp, i64, i64, vp, sz]),
        "mq_unpack": (ctypes.c_int, [ctypes.c_int, vp, i64, i64, vp]),
        "mq_unpack_device": (ctypes.c_int, [ctypes.c_int, vp, i64, i64, vp, vp]),
        "moe_quant_workspace_size": (sz, [cfgp, i32]),
        "moe_quant_forward": (ctypes.c_int, [cfgp, i32, vp, vp, vp, ctypes.POINTER(mq_expert_table), vp,
                                             vp, vp, vp, vp, sz, vp]),
        "moe_quant_forward_noalloc": (ctypes.c_int, [cfgp, i32, vp, vp, vp, ctypes.POINTER(mq_expert_table), vp,
                                                     vp, vp, vp, vp]),
        "moe_quant_route": (ctypes.c_int, [cfgp, i32, vp, vp, vp, vp, vp, vp, vp, vp, vp, sz, vp]),
        "moe_quant_status": (ctypes.c_int, [cfgp, i32, vp, sz, ctypes.POINTER(ctypes.c_uint32), vp]),
        "moe_quant_status_noalloc": (ctypes.c_int, [cfgp, i32, ctypes.POINTER(ctypes.c_uint32), vp]),
        "mq_strerror": (ctypes.c_char_p, [ctypes.c_int]),
        "mq_set_path": (ctypes.c_int, [ctypes.c_int, i32]),
        "mq_test_fail_next_decode": (ctypes.c_int, [ctypes.c_uint64]),
        "mq_profile_enable": (ctypes.c_int, [i32]),
        "mq_profile_collect": (ctypes.c_int, [ctypes.POINTER(mq_kernel_stat), i32]),
        "mq_plan_precision": (ctypes.c_int, [ctypes.POINTER(mq_plan_cfg), ctypes.POINTER(mq_plan_tensor), i32, vp,
                                             ctypes.POINTER(ctypes.c_int64)]),
        "mq_binary_partition_order": (ctypes.c_int, [i32, vp]),
        "mq_expert_importance": (ctypes.c_int, [vp, vp, i32, i32, i32, ctypes.c_double, ctypes.c_double, vp, vp,
                                                ctypes.POINTER(ctypes.c_int32)]),
        "mq_activation_plan": (ctypes.c_int, [i32, ctypes.c_double, i32, vp, i64, vp, ctypes.POINTER(ctypes.c_int64)]),
        "mq_expert_stats_bytes": (sz, [i32]),
        "mq_expert_stats_reset": (ctypes.c_int, [vp, i32, vp]),
        "mq_expert_stats_add": (ctypes.c_int, [vp, i32, vp, vp, i32, i32, vp]),
        "mq_expert_stats_scores": (ctypes.c_int, [vp, i32, ctypes.c_double, ctypes.c_double, vp, vp, vp, vp,
                                                  ctypes.POINTER(ctypes.c_int32), vp]),
    }
    for name, (res, args) in sig.items():
        fn = getattr(L, name)
        fn.restype, fn.argtypes = res, args
    return L


_lib = _load()
EXPORTED = ("mq_packed_size", "mq_pack", "mq_unpack", "mq_unpack_device", "moe_quant_workspace_size",
            "moe_quant_forward", "moe_quant_forward_noalloc", "moe_quant_route", "mq_strerror", "mq_set_path", "mq_profile_enable",
            "mq_profile_collect", "mq_plan_precision", "mq_binary_partition_order", "moe_quant_status",
            "moe_quant_status_noalloc", "mq_expert_importance", "mq_test_fail_next_decode",
            "mq_activation_plan", "mq_expert_stats_bytes", "mq_expert_stats_reset", "mq_expert_stats_add", "mq_expert_stats_scores")


def _ptr(a):
    """Data pointer of a torch tensor / numpy array / int / None."""
    if a is None:
        return None
    if isinstance(a, int):
        return a
    if hasattr(a, "data_ptr"):
        return a.data_ptr()
    return a.ctypes.data


def _stream(stream):
    if stream is None:
        try:
            import torch
            if torch.cuda.is_available():
                return torch.cuda.current_stream().cuda_stream
        except ImportError:
            pass
        return None
    return getattr(stream, "cuda_stream", stream)


def _check(fn, rc):
    if rc != MQ_OK:
        raise MoeqError(fn, rc)
    return rc


def _fmt(f):
    return FORMATS[f] if isinstance(f, str) else int(f)


def mq_strerror(status: int) -> str:
    return _lib.mq_strerror(status).decode()


def mq_packed_size(fmt, rows: int, cols: int) -> int:
    return int(_lib.mq_packed_size(_fmt(fmt), rows, cols))


def mq_pack(fmt, w, dst=None):
    """Host quantizer. w: float32 [rows, cols] (numpy or CPU tensor).
    Returns dst (a new numpy uint8 array when dst is None)."""
    import numpy as np
    w = np.ascontiguousarray(w if not hasattr(w, "numpy") else w.numpy(), dtype=np.float32)
    rows, cols = w.shape
    n = mq_packed_size(fmt, rows, cols)
    if dst is None:
        dst = np.empty(n, np.uint8)
    _check("mq_pack", _lib.mq_pack(_fmt(fmt), w.ctypes.data, rows, cols, _ptr(dst), _nbytes(dst)))
    return dst


def _nbytes(a) -> int:
    if hasattr(a, "element_size"):
        return a.numel() * a.element_size()
    return a.nbytes


def _need(fn, a, n):
    """The C entry points take no source/destination sizes: refuse buffers
    smaller than the tensor they describe before passing their pointers."""
    if a is not None and not isinstance(a, int) and _nbytes(a) < n:
        raise MoeqError(fn, MQ_EINVAL)


def mq_unpack(fmt, src, rows: int, cols: int):
    import numpy as np
    src = np.ascontiguousarray(src, dtype=np.uint8)
    _need("mq_unpack", src, mq_packed_size(fmt, rows, cols))
    out = np.empty((rows, cols), np.float32)
    _check("mq_unpack", _lib.mq_unpack(_fmt(fmt), src.ctypes.data, rows, cols, out.ctypes.data))
    return out


def mq_unpack_device(fmt, src, rows: int, cols: int, dst, stream=None):
    _need("mq_unpack_device", src, mq_packed_size(fmt, rows, cols))
    _need("mq_unpack_device", dst, 4 * max(rows, 0) * max(cols, 0))
    _check("mq_unpack_device",
           _lib.mq_unpack_device(_fmt(fmt), _ptr(src), rows, cols, _ptr(dst), _stream(stream)))
    return dst


def make_cfg(hidden, inter, n_experts, n_groups, topk_group, top_k, routed_scale=1.0, has_shared=False):
    return mq_layer_cfg(hidden, inter, n_experts, n_groups, topk_group, top_k, float(routed_scale),
                        int(bool(has_shared)))


def moe_quant_workspace_size(cfg: mq_layer_cfg, n_tokens: int) -> int:
    return int(_lib.moe_quant_workspace_size(ctypes.byref(cfg), n_tokens))


class ExpertTable:
    """Holds the ctypes expert table built from per-expert (gate, up, down)
    device tensors or raw pointers; keeps the ctypes arrays alive."""

    def __init__(self, experts, shared=None):
        n = len(experts)
        self._arr = (mq_expert_weights * max(n, 1))()
        for i, (g, u, d) in enumerate(experts):
            self._arr[i] = mq_expert_weights(_ptr(g), _ptr(u), _ptr(d))
        self._shared = None
        if shared is not None:
            self._shared = mq_expert_weights(*[_ptr(t) for t in shared])
        self.table = mq_expert_table(
            ctypes.cast(self._arr, ctypes.POINTER(mq_expert_weights)),
            ctypes.pointer(self._shared) if self._shared is not None else None)


def moe_quant_forward(cfg, n_tokens, x, router_w, bias, expert_table: ExpertTable, fmt_per_tensor, out,
                      topk_idx=None, topk_w=None, workspace=None, ws_bytes=None, stream=None):
    import numpy as np
    fmt = np.ascontiguousarray(fmt_per_tensor, dtype=np.uint8).reshape(-1)
    if ws_bytes is None:
        ws_bytes = workspace.numel() * workspace.element_size() if workspace is not None else 0
    rc = _lib.moe_quant_forward(ctypes.byref(cfg), n_tokens, _ptr(x), _ptr(router_w), _ptr(bias),
                                ctypes.byref(expert_table.table), fmt.ctypes.data, _ptr(out), _ptr(topk_idx),
                                _ptr(topk_w), _ptr(workspace), ws_bytes, _stream(stream))
    return _check("moe_quant_forward", rc)


def moe_quant_forward_noalloc(cfg, n_tokens, x, router_w, bias, expert_table: ExpertTable, fmt_per_tensor, out,
                              topk_idx=None, topk_w=None, stream=None):
    """moe_quant_forward with the library's fixed 16 MiB device scratch instead
    of a caller workspace (nothing is allocated)."""
    import numpy as np
    fmt = np.ascontiguousarray(fmt_per_tensor, dtype=np.uint8).reshape(-1)
    rc = _lib.moe_quant_forward_noalloc(ctypes.byref(cfg), n_tokens, _ptr(x), _ptr(router_w), _ptr(bias),
                                        ctypes.byref(expert_table.table), fmt.ctypes.data, _ptr(out),
                                        _ptr(topk_idx), _ptr(topk_w), _stream(stream))
    return _check("moe_quant_forward_noalloc", rc)


def moe_quant_route(cfg, n_tokens, x, router_w, bias, topk_idx, topk_w, offsets=None, perm=None, inv=None,
                    workspace=None, ws_bytes=None, stream=None):
    if ws_bytes is None:
        ws_bytes = workspace.numel() * workspace.element_size() if workspace is not None else 0
    rc = _lib.moe_quant_route(ctypes.byref(cfg), n_tokens, _ptr(x), _ptr(router_w), _ptr(bias), _ptr(topk_idx),
                              _ptr(topk_w), _ptr(offsets), _ptr(perm), _ptr(inv), _ptr(workspace), ws_bytes,
                              _stream(stream))
    return _check("moe_quant_route", rc)


def moe_quant_status(cfg, n_tokens, workspace, ws_bytes=None, stream=None) -> int:
    """Error bits of the last forward call with this workspace (0 = none);
    raises MoeqError on bad arguments.  Waits for the stream."""
    if ws_bytes is None:
        ws_bytes = workspace.numel() * workspace.element_size() if workspace is not None else 0
    bits = ctypes.c_uint32(0)
    rc = _lib.moe_quant_status(ctypes.byref(cfg), n_tokens, _ptr(workspace), ws_bytes, ctypes.byref(bits),
                               _stream(stream))
    if rc not in (MQ_OK, MQ_EDEVICE):
        raise MoeqError("moe_quant_status", rc)
    return int(bits.value)


def moe_quant_status_noalloc(cfg, n_tokens, stream=None) -> int:
    bits = ctypes.c_uint32(0)
    rc = _lib.moe_quant_status_noalloc(ctypes.byref(cfg), n_tokens, ctypes.byref(bits), _stream(stream))
    if rc not in (MQ_OK, MQ_EDEVICE):
        raise MoeqError("moe_quant_status_noalloc", rc)
    return int(bits.value)


def mq_test_fail_next_decode(wait_ns: int):
    """Test hook: the next decode call's pipeline waits give up after wait_ns
    (the gate/up producer posts nothing for its first stage)."""
    return _check("mq_test_fail_next_decode", _lib.mq_test_fail_next_decode(int(wait_ns)))


def mq_set_path(mode: int, prefill_threshold: int = 0):
    return _check("mq_set_path", _lib.mq_set_path(mode, prefill_threshold))


def mq_profile_enable(max_launches: int):
    return _check("mq_profile_enable", _lib.mq_profile_enable(max_launches))


def mq_profile_collect(max_entries: int = 64):
    arr = (mq_kernel_stat * max_entries)()
    n = _lib.mq_profile_collect(arr, max_entries)
    return [(arr[i].name.decode(), int(arr[i].launches), float(arr[i].total_ms)) for i in range(n)]


# ------------------------------------------------------------ planner ---
MQ_TENSOR_OTHER, MQ_TENSOR_EXPERT_GATE, MQ_TENSOR_EXPERT_UP, MQ_TENSOR_EXPERT_DOWN = 0, 1, 2, 3


def mq_plan_precision(tensors, bits64, low, lowest, small_level, medium_level, floor_level, small_max, medium_max,
                      mem_limit_bytes):
    """tensors: sequence of (params, layer, kind, sens).  Returns (levels as a
    numpy int32 array, total bits in 1/64-bit units)."""
    import numpy as np
    n = len(tensors)
    arr = (mq_plan_tensor * max(n, 1))()
    for i, (p, ly, k, s) in enumerate(tensors):
        arr[i] = mq_plan_tensor(int(p), int(ly), int(k), float(s))
    b = (ctypes.c_int32 * len(bits64))(*[int(v) for v in bits64])
    cfg = mq_plan_cfg(len(bits64), b, low, lowest, small_level, medium_level, floor_level, int(small_max),
                      int(medium_max), int(mem_limit_bytes))
    out = np.empty(max(n, 1), np.int32)
    total = ctypes.c_int64(0)
    _check("mq_plan_precision", _lib.mq_plan_precision(ctypes.byref(cfg), arr, n, out.ctypes.data, ctypes.byref(total)))
    return out[:n], int(total.value)


def mq_binary_partition_order(n: int):
    import numpy as np
    out = np.empty(max(n, 1), np.int32)
    _check("mq_binary_partition_order", _lib.mq_binary_partition_order(n, out.ctypes.data))
    return out[:n]


def mq_expert_importance(topk_idx, topk_w, n_experts: int, alpha: float = 0.5, retain: float = 0.75):
    """Host arrays [n_tokens, top_k] (numpy or CPU tensors).  Returns (kept
    expert ids ascending, I_e scores)."""
    import numpy as np
    idx = np.ascontiguousarray(topk_idx.numpy() if hasattr(topk_idx, "numpy") else topk_idx, dtype=np.int32)
    w = np.ascontiguousarray(topk_w.numpy() if hasattr(topk_w, "numpy") else topk_w, dtype=np.float32)
    if idx.ndim != 2 or w.shape != idx.shape:
        raise MoeqError("mq_expert_importance", MQ_EINVAL)
    scores = np.empty(max(n_experts, 1), np.float64)
    keep = np.empty(max(n_experts, 1), np.int32)
    nk = ctypes.c_int32(0)
    _check("mq_expert_importance",
           _lib.mq_expert_importance(idx.ctypes.data, w.ctypes.data, idx.shape[0], idx.shape[1], n_experts,
                                     float(alpha), float(retain), scores.ctypes.data, keep.ctypes.data,
                                     ctypes.byref(nk)))
    return keep[:nk.value], scores[:n_experts]


def mq_activation_plan(k_orig: int, retain: float, params_per_expert, flops_budget: int):
    """Per-layer activated experts k_i and the plan's FLOPs_active (Sec. 3.2)."""
    import numpy as np
    P = np.ascontiguousarray(np.asarray(params_per_expert, dtype=np.int64).reshape(-1))
    k = np.empty(max(P.size, 1), np.int32)
    fl = ctypes.c_int64(0)
    _check("mq_activation_plan", _lib.mq_activation_plan(int(k_orig), float(retain), int(P.size), P.ctypes.data,
                                                         int(flops_budget), k.ctypes.data, ctypes.byref(fl)))
    return k[:P.size], int(fl.value)


# ------------------------------------------- device expert statistics ---
def mq_expert_stats_bytes(n_experts: int) -> int:
    return int(_lib.mq_expert_stats_bytes(n_experts))


def mq_expert_stats_reset(stats, n_experts: int, stream=None):
    _need("mq_expert_stats_reset", stats, mq_expert_stats_bytes(n_experts))
    return _check("mq_expert_stats_reset", _lib.mq_expert_stats_reset(_ptr(stats), n_experts, _stream(stream)))


def mq_expert_stats_add(stats, n_experts: int, topk_idx, topk_w, n_tokens: int, top_k: int, stream=None):
    """stats: device buffer of mq_expert_stats_bytes(n_experts) bytes;
    topk_idx / topk_w: device int32 / fp32 [n_tokens, top_k]."""
    _need("mq_expert_stats_add", stats, mq_expert_stats_bytes(n_experts))
    if n_tokens > 0:
        _need("mq_expert_stats_add", topk_idx, 4 * n_tokens * top_k)
        _need("mq_expert_stats_add", topk_w, 4 * n_tokens * top_k)
    return _check("mq_expert_stats_add", _lib.mq_expert_stats_add(_ptr(stats), n_experts, _ptr(topk_idx),
                                                                  _ptr(topk_w), n_tokens, top_k, _stream(stream)))


def mq_expert_stats_scores(stats, n_experts: int, alpha: float, retain: float, freq=None, mean_w=None, scores=None,
                           keep=None, stream=None) -> int:
    """Writes the requested device outputs; returns ceil(retain n_experts),
    the number of ids written to keep."""
    _need("mq_expert_stats_scores", stats, mq_expert_stats_bytes(n_experts))
    nk = ctypes.c_int32(0)
    # no outputs: only the kept count, nothing enqueued
    _check("mq_expert_stats_scores", _lib.mq_expert_stats_scores(_ptr(stats), n_experts, float(alpha), float(retain),
                                                                 None, None, None, None, ctypes.byref(nk), None))
    for a in (freq, mean_w, scores):
        if a is not None:
            _need("mq_expert_stats_scores", a, 8 * n_experts)
    if keep is not None:
        _need("mq_expert_stats_scores", keep, 4 * nk.value)
    _check("mq_expert_stats_scores",
           _lib.mq_expert_stats_scores(_ptr(stats), n_experts, float(alpha), float(retain), _ptr(freq), _ptr(mean_w),
                                       _ptr(scores), _ptr(keep), None, _stream(stream)))
    return int(nk.value)
