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
every size and checksum and raises ValueError on a mismatch, so a truncated
or corrupted file never reaches the kernels.
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
    fm = np.asarray(header["formats"], np.uint8).reshape(-1, 3)
    E = int(cfg["n_experts"])
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
    out["bias"] = conv(got["bias"].view(np.float32)) if "bias" in got else None

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
