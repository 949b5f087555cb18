"""Save and load a packed MoE layer: the planar streams as raw bytes plus a
JSON header.

The forward pass is stateless, so a layer's packed tensors, its router and
its per-tensor formats are its whole state.  A checkpoint directory holds

  layer.json   {"version": 1, "cfg": {...mq_layer_cfg fields...},
                "formats": [[gate, up, down], ...]  (routed experts, then shared),
                "streams": [{"name", "file", "offset", "bytes", "sha256"}, ...]}
  layer.bin    every stream at a 256-byte aligned offset

Streams: "router_w" (fp32 [E, H]), "bias" (fp32 [E], optional), and
"e{i}.gate|up|down" / "shared.gate|up|down" (packed bytes, sizes checked
against mq_packed_size for the stream's format and shape).  Loading checks
the configuration's bounds, the formats table (one row per expert, known
codes), every size and checksum and raises ValueError on a mismatch, so a
truncated, corrupted or inconsistent file never reaches the kernels.
"""
from __future__ import annotations

import hashlib
import json
import os

import numpy as np

from . import mq_packed_size

VERSION = 1
_ALIGN = 256
_CFG_FIELDS = ("hidden", "inter", "n_experts", "n_groups", "topk_group", "top_k", "routed_scale", "has_shared")


def _check_cfg(cfg: dict) -> None:
    """The mq_layer_cfg bounds moe_quant_forward enforces, as ValueError."""
    missing = [k for k in _CFG_FIELDS if k not in cfg]
    if missing:
        raise ValueError(f"cfg: missing fields {missing}")
    try:
        H, I, E, G, Gk, K, S = (int(cfg[k]) for k in _CFG_FIELDS if k != "routed_scale")
        rs = float(cfg["routed_scale"])
    except (TypeError, ValueError) as exc:
        raise ValueError(f"cfg: non-numeric field ({exc})") from None
    checks = [
        (128 <= H <= 32768 and H % 128 == 0, "hidden must be a multiple of 128 in [128, 32768]"),
        (128 <= I <= 16384 and I % 128 == 0, "inter must be a multiple of 128 in [128, 16384]"),
        (1 <= E <= 256, "n_experts must be in [1, 256]"),
        (1 <= G <= 64 and E % G == 0, "n_groups must be in [1, 64] and divide n_experts"),
        (1 <= Gk <= G, "topk_group must be in [1, n_groups]"),
        (1 <= K <= 32 and K <= Gk * (E // G), "top_k must be in [1, 32] and at most topk_group * n_experts / n_groups"),
        (S in (0, 1), "has_shared must be 0 or 1"),
        (np.isfinite(rs), "routed_scale must be finite"),
    ]
    for ok, msg in checks:
        if not ok:
            raise ValueError(f"cfg: {msg}")


def _valid_format(f: int) -> bool:
    """A format code the library knows (it sizes a tensor in it)."""
    return mq_packed_size(int(f), 32, 256) > 0


def _host(a) -> np.ndarray:
    if hasattr(a, "detach"):
        a = a.detach().cpu().numpy()
    return np.ascontiguousarray(a)


def _shapes(cfg: dict):
    H, I = cfg["hidden"], cfg["inter"]
    return {"gate": (I, H), "up": (I, H), "down": (H, I)}


def save_layer(path: str, cfg: dict, formats, experts, shared=None, router_w=None, bias=None) -> None:
    """cfg: dict of mq_layer_cfg fields; formats: uint8 [(E + has_shared), 3];
    experts: E triples of packed (gate, up, down) byte arrays (numpy or
    tensors, host or device); shared: one triple or None; router_w: fp32
    [E, H]; bias: fp32 [E] or None."""
    cfg = {k: (float(cfg[k]) if k == "routed_scale" else int(cfg[k])) for k in _CFG_FIELDS}
    E = cfg["n_experts"]
    fm = np.asarray(formats, np.uint8).reshape(-1, 3)
    if fm.shape[0] != E + cfg["has_shared"] or len(experts) != E or (shared is None) == bool(cfg["has_shared"]):
        raise ValueError("formats / experts / shared do not match the configuration")
    if router_w is None:
        raise ValueError("router_w is required")
    shp = _shapes(cfg)
    streams = [("router_w", _host(router_w).astype(np.float32, copy=False), (E, cfg["hidden"]), None)]
    if bias is not None:
        streams.append(("bias", _host(bias).astype(np.float32, copy=False), (E,), None))
    owners = [(f"e{i}", t, fm[i]) for i, t in enumerate(experts)]
    if shared is not None:
        owners.append(("shared", shared, fm[E]))
    for name, trip, f in owners:
        for j, part in enumerate(("gate", "up", "down")):
            streams.append((f"{name}.{part}", _host(trip[j]).view(np.uint8).reshape(-1), shp[part], int(f[j])))
    os.makedirs(path, exist_ok=True)
    header = {"version": VERSION, "cfg": cfg, "formats": fm.tolist(), "streams": []}
    off = 0
    with open(os.path.join(path, "layer.bin"), "wb") as fb:
        for name, arr, shape, fmt in streams:
            raw = arr.tobytes()
            if fmt is not None and len(raw) != mq_packed_size(fmt, *shape):
                raise ValueError(f"{name}: {len(raw)} bytes, format {fmt} {shape} needs {mq_packed_size(fmt, *shape)}")
            if fmt is None and arr.size != int(np.prod(shape)):
                raise ValueError(f"{name}: shape {arr.shape}, expected {shape}")
            pad = (-off) % _ALIGN
            fb.write(b"\0" * pad)
            off += pad
            fb.write(raw)
            header["streams"].append({"name": name, "file": "layer.bin", "offset": off, "bytes": len(raw),
                                      "shape": list(shape), "format": fmt,
                                      "sha256": hashlib.sha256(raw).hexdigest()})
            off += len(raw)
    with open(os.path.join(path, "layer.json"), "w") as fj:
        json.dump(header, fj, indent=1)


def load_layer(path: str, device=None) -> dict:
    """Returns {"cfg", "formats", "router_w", "bias", "experts", "shared"}
    with numpy arrays, or torch tensors on `device` when it is given."""
    with open(os.path.join(path, "layer.json")) as fj:
        header = json.load(fj)
    if header.get("version") != VERSION:
        raise ValueError(f"unsupported checkpoint version {header.get('version')}")
    cfg = header["cfg"]
    _check_cfg(cfg)
    fm = np.asarray(header["formats"], np.int64)
    E = int(cfg["n_experts"])
    n_rows = E + int(cfg["has_shared"])
    if fm.ndim != 2 or fm.shape != (n_rows, 3):
        raise ValueError(f"formats: shape {fm.shape}, the configuration needs ({n_rows}, 3)")
    bad = sorted({int(f) for f in fm.reshape(-1) if not _valid_format(int(f))})
    if bad:
        raise ValueError(f"formats: unknown format codes {bad}")
    fm = fm.astype(np.uint8)
    shp = _shapes(cfg)
    blob = np.fromfile(os.path.join(path, "layer.bin"), np.uint8)
    got = {}
    for s in header["streams"]:
        o, n = int(s["offset"]), int(s["bytes"])
        if o % _ALIGN or o + n > blob.size:
            raise ValueError(f"{s['name']}: stream outside the file (truncated?)")
        raw = blob[o:o + n]
        if hashlib.sha256(raw.tobytes()).hexdigest() != s["sha256"]:
            raise ValueError(f"{s['name']}: checksum mismatch")
        got[s["name"]] = raw
    out = {"cfg": cfg, "formats": fm}

    def conv(a):
        if device is None:
            return a.copy()
        import torch
        return torch.from_numpy(a.copy()).to(device)

    if "router_w" not in got:
        raise ValueError("router_w missing")
    rw = got["router_w"].view(np.float32)
    if rw.size != E * int(cfg["hidden"]):
        raise ValueError("router_w size does not match the configuration")
    out["router_w"] = conv(rw.reshape(E, int(cfg["hidden"])))
    if "bias" in got:
        b = got["bias"].view(np.float32)
        if b.size != E:
            raise ValueError(f"bias: {b.size} values, the configuration has {E} experts")
        out["bias"] = conv(b)
    else:
        out["bias"] = None

    def trip(name, row):
        parts = []
        for j, part in enumerate(("gate", "up", "down")):
            key = f"{name}.{part}"
            if key not in got:
                raise ValueError(f"{key} missing")
            need = mq_packed_size(int(row[j]), *shp[part])
            if got[key].size != need:
                raise ValueError(f"{key}: {got[key].size} bytes, format {int(row[j])} needs {need}")
            parts.append(conv(got[key]))
        return tuple(parts)

    out["experts"] = [trip(f"e{i}", fm[i]) for i in range(E)]
    out["shared"] = trip("shared", fm[E]) if int(cfg["has_shared"]) else None
    return out
