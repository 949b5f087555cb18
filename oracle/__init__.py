"""Oracle for the quantized MoE expert FFN — TEST INFRASTRUCTURE ONLY.

A thin ctypes wrapper around ``oracle.c`` (plain single-threaded C,
``-ffp-contract=off``).  Only ``tests/``, ``__graft_entry__.smoke()`` and the
benchmark's CPU-baseline leg may import this package; the product library
(``paper_2509_25689_gb300``) never does, and this package never imports it.
"""
from __future__ import annotations

import ctypes
import os
import platform
import subprocess

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SO = os.path.join(_HERE, f"liboracle_{platform.machine()}.so")
# the same source built with -fopenmp: independent rows and tokens split over
# threads, identical arithmetic per row/token (OMP_NUM_THREADS sets the count)
_SO_OMP = os.path.join(_HERE, f"liboracle_omp_{platform.machine()}.so")

Q2_K, Q3_K, Q4_K, Q8_0, Q6_K, BF16 = 1, 2, 3, 4, 5, 6
FORMATS = {"Q2_K": Q2_K, "Q3_K": Q3_K, "Q4_K": Q4_K, "Q8_0": Q8_0, "Q6_K": Q6_K, "BF16": BF16}


class OracleLayer(ctypes.Structure):
    _fields_ = [
        ("hidden", ctypes.c_int32), ("inter", ctypes.c_int32),
        ("n_experts", ctypes.c_int32), ("n_groups", ctypes.c_int32),
        ("topk_group", ctypes.c_int32), ("top_k", ctypes.c_int32),
        ("routed_scale", ctypes.c_float), ("has_shared", ctypes.c_int32),
    ]


def build(force: bool = False) -> str:
    """Compile oracle.c into liboracle.so (gcc, no fast-math, no contraction),
    and the OpenMP build of the same source."""
    src = os.path.join(_HERE, "oracle.c")
    newest = max(os.path.getmtime(src), os.path.getmtime(os.path.join(_HERE, "oracle.h")))
    for so, extra in ((_SO, []), (_SO_OMP, ["-fopenmp"])):
        if not force and os.path.exists(so) and os.path.getmtime(so) >= newest:
            continue
        tmp = so + f".tmp{os.getpid()}"
        subprocess.check_call(["gcc", "-O1", "-std=c11", "-ffp-contract=off", "-fno-fast-math", *extra,
                               "-fPIC", "-shared", "-o", tmp, src, "-lm"])
        os.replace(tmp, so)
    return _SO


_libs = {}
_omp = False


def use_openmp(on: bool) -> None:
    """Route the following calls to the OpenMP build (True) or the plain
    single-threaded build (False, the default)."""
    global _omp
    _omp = bool(on)


def lib():
    key = _omp
    if key not in _libs:
        build()
        L = ctypes.CDLL(_SO_OMP if key else _SO)
        vp, i64, i32 = ctypes.c_void_p, ctypes.c_int64, ctypes.c_int32
        L.oracle_packed_size.restype = ctypes.c_size_t
        L.oracle_packed_size.argtypes = [ctypes.c_int, i64, i64]
        L.oracle_pack.restype = ctypes.c_int
        L.oracle_pack.argtypes = [ctypes.c_int, vp, i64, i64, vp, ctypes.c_size_t]
        L.oracle_unpack.restype = ctypes.c_int
        L.oracle_unpack.argtypes = [ctypes.c_int, vp, i64, i64, vp]
        L.oracle_sigmoid.restype = ctypes.c_float
        L.oracle_sigmoid.argtypes = [ctypes.c_float]
        L.oracle_router_logit.restype = ctypes.c_float
        L.oracle_router_logit.argtypes = [vp, vp, i32]
        L.oracle_route.restype = ctypes.c_int
        L.oracle_route.argtypes = [ctypes.POINTER(OracleLayer), i32, vp, vp, vp, vp, vp, vp, vp]
        L.oracle_select.restype = ctypes.c_int
        L.oracle_select.argtypes = [ctypes.POINTER(OracleLayer), i32, vp, vp, vp, vp]
        L.oracle_permute.restype = ctypes.c_int
        L.oracle_permute.argtypes = [i32, i32, i32, vp, vp, vp, vp]
        L.oracle_moe_forward.restype = ctypes.c_int
        L.oracle_moe_forward.argtypes = [ctypes.POINTER(OracleLayer), i32, vp, vp, vp,
                                         vp, vp, vp, vp, vp, vp, vp]
        _libs[key] = L
    return _libs[key]


def _p(a: np.ndarray | None):
    return None if a is None else a.ctypes.data_as(ctypes.c_void_p)


def _fmt(f) -> int:
    return FORMATS[f] if isinstance(f, str) else int(f)


def packed_size(fmt, rows: int, cols: int) -> int:
    return int(lib().oracle_packed_size(_fmt(fmt), rows, cols))


def pack(fmt, w: np.ndarray) -> np.ndarray:
    w = np.ascontiguousarray(w, dtype=np.float32)
    rows, cols = w.shape
    out = np.zeros(packed_size(fmt, rows, cols), dtype=np.uint8)
    rc = lib().oracle_pack(_fmt(fmt), _p(w), rows, cols, _p(out), out.nbytes)
    if rc:
        raise ValueError(f"oracle_pack failed ({rc})")
    return out


def unpack(fmt, packed: np.ndarray, rows: int, cols: int) -> np.ndarray:
    packed = np.ascontiguousarray(packed, dtype=np.uint8)
    if packed.nbytes < packed_size(fmt, rows, cols):
        raise ValueError("packed buffer too small")
    out = np.empty((rows, cols), dtype=np.float32)
    if lib().oracle_unpack(_fmt(fmt), _p(packed), rows, cols, _p(out)):
        raise ValueError("oracle_unpack failed")
    return out


def sigmoid(z: float) -> float:
    return float(lib().oracle_sigmoid(float(z)))


def router_logit(x_bits: np.ndarray, w: np.ndarray) -> float:
    x_bits = np.ascontiguousarray(x_bits, dtype=np.uint16)
    w = np.ascontiguousarray(w, dtype=np.float32)
    return float(lib().oracle_router_logit(_p(x_bits), _p(w), x_bits.shape[-1]))


def make_layer(hidden, inter, n_experts, n_groups, topk_group, top_k,
               routed_scale=1.0, has_shared=False) -> OracleLayer:
    return OracleLayer(hidden, inter, n_experts, n_groups, topk_group, top_k,
                       float(routed_scale), int(bool(has_shared)))


def route(layer: OracleLayer, x_bits: np.ndarray, router_w: np.ndarray,
          bias: np.ndarray | None):
    """Returns idx [T,k] int32, w [T,k] f32, z [T,E] f32, s [T,E] f32."""
    x_bits = np.ascontiguousarray(x_bits, dtype=np.uint16)
    router_w = np.ascontiguousarray(router_w, dtype=np.float32)
    T = x_bits.shape[0]
    E, K = layer.n_experts, layer.top_k
    idx = np.zeros((T, K), np.int32)
    w = np.zeros((T, K), np.float32)
    z = np.zeros((T, E), np.float32)
    s = np.zeros((T, E), np.float32)
    b = None if bias is None else np.ascontiguousarray(bias, dtype=np.float32)
    if lib().oracle_route(ctypes.byref(layer), T, _p(x_bits), _p(router_w), _p(b),
                          _p(idx), _p(w), _p(z), _p(s)):
        raise ValueError("oracle_route failed")
    return idx, w, z, s


def select(layer: OracleLayer, s: np.ndarray, bias: np.ndarray | None):
    """The selection step alone on precomputed sigmoid scores s [T, E]:
    returns idx [T,k] int32, w [T,k] f32 (identical to route's for the same
    scores and bias)."""
    s = np.ascontiguousarray(s, dtype=np.float32)
    T = s.shape[0]
    K = layer.top_k
    idx = np.zeros((T, K), np.int32)
    w = np.zeros((T, K), np.float32)
    b = None if bias is None else np.ascontiguousarray(bias, dtype=np.float32)
    if lib().oracle_select(ctypes.byref(layer), T, _p(s), _p(b), _p(idx), _p(w)):
        raise ValueError("oracle_select failed")
    return idx, w


def permute(idx: np.ndarray, n_experts: int):
    idx = np.ascontiguousarray(idx, dtype=np.int32)
    T, K = idx.shape
    offsets = np.zeros(n_experts + 1, np.int32)
    perm = np.zeros(T * K, np.int32)
    inv = np.zeros(T * K, np.int32)
    if lib().oracle_permute(T, K, n_experts, _p(idx), _p(offsets), _p(perm), _p(inv)):
        raise ValueError("oracle_permute failed")
    return offsets, perm, inv


def moe_forward(layer: OracleLayer, x_bits: np.ndarray, router_w: np.ndarray,
                bias: np.ndarray | None, gate: list, up: list, down: list,
                fmt: np.ndarray):
    """Full layer on host arrays.  gate/up/down: lists of packed uint8 arrays
    (routed experts then, if layer.has_shared, the shared expert); fmt:
    uint8 [(E+shared), 3].  Returns y [T,H] f32, idx, w."""
    x_bits = np.ascontiguousarray(x_bits, dtype=np.uint16)
    router_w = np.ascontiguousarray(router_w, dtype=np.float32)
    T = x_bits.shape[0]
    H, K = layer.hidden, layer.top_k
    n = layer.n_experts + (1 if layer.has_shared else 0)
    assert len(gate) == len(up) == len(down) == n
    keep = [np.ascontiguousarray(a, dtype=np.uint8) for a in (*gate, *up, *down)]
    ptr_t = ctypes.c_void_p * n
    gp = ptr_t(*[a.ctypes.data for a in keep[:n]])
    upp = ptr_t(*[a.ctypes.data for a in keep[n:2 * n]])
    dp = ptr_t(*[a.ctypes.data for a in keep[2 * n:]])
    fmt = np.ascontiguousarray(fmt, dtype=np.uint8).reshape(-1)
    y = np.zeros((T, H), np.float32)
    idx = np.zeros((T, K), np.int32)
    w = np.zeros((T, K), np.float32)
    b = None if bias is None else np.ascontiguousarray(bias, dtype=np.float32)
    rc = lib().oracle_moe_forward(ctypes.byref(layer), T, _p(x_bits), _p(router_w), _p(b),
                                  ctypes.cast(gp, ctypes.c_void_p), ctypes.cast(upp, ctypes.c_void_p),
                                  ctypes.cast(dp, ctypes.c_void_p), _p(fmt), _p(y), _p(idx), _p(w))
    if rc:
        raise ValueError("oracle_moe_forward failed")
    return y, idx, w
