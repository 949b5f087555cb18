"""Pins for the oracle's block formats (pack / unpack).

The expert tensors are stored in k-quant style block formats (Sec. 3.3,
Q2_K/Q3_K/Q4_K/Q6_K and Q8 types, and bf16 for tensors kept unquantized;
Sec. 4.1).  These tests tie the oracle to
facts that do not come from its own code: hand-built blocks with values
worked out by hand, exact round trips of blocks that lie on the grid,
the nearest-grid-point property, and a closed-form error bound.
"""
import json
import os

import numpy as np
import pytest

HERE = os.path.dirname(os.path.abspath(__file__))
FMTS = ["Q2_K", "Q3_K", "Q4_K", "Q8_0", "Q6_K", "BF16"]


def _cases():
    with open(os.path.join(HERE, "golden", "hand_blocks.json")) as f:
        return json.load(f)["cases"]


@pytest.mark.parametrize("case", _cases(), ids=lambda c: c["name"])
def test_hand_built_blocks(orc, case):
    rows, cols = case["rows"], case["cols"]
    assert orc.packed_size(case["format"], rows, cols) == case["size"]
    buf = np.zeros(case["size"], np.uint8)
    for off, val in case["bytes"].items():
        buf[int(off)] = val
    got = orc.unpack(case["format"], buf, rows, cols).reshape(-1)
    want = np.full(rows * cols, case["expect_default"], np.float32)
    for a, b, v in case["expect_ranges"]:
        want[a:b] = v
    for k, v in case["expect"].items():
        want[int(k)] = v
    np.testing.assert_array_equal(got, want)


@pytest.mark.parametrize("fmt,rows,cols,nominal", [
    ("Q2_K", 2048, 7168, 4816896),    # V3 gate/up in Q2_K style
    ("Q3_K", 7168, 2048, 6307840),    # V3 down in Q3_K style
    ("Q4_K", 2048, 7168, 8257536),    # 144 B / 256 weights
    ("Q8_0", 2048, 7168, 15597568),   # 34 B / 32 weights
    ("Q6_K", 2048, 7168, 12042240),   # 210 B / 256 weights
    ("BF16", 2048, 7168, 29360128),   # 2 B / weight
    ("Q4_K", 128, 256, 18432),        # tiny gate/up
    ("Q4_K", 256, 128, 36864),        # tiny down: row padded to one block
])
def test_sizes_match_nominal_bits_per_weight(orc, fmt, rows, cols, nominal):
    assert orc.packed_size(fmt, rows, cols) == nominal


def test_all_zero_weights_pack_to_zero(orc):
    w = np.zeros((3, 300), np.float32)
    for f in FMTS:
        p = orc.pack(f, w)
        # Q3_K stores sub-scales and codes with an offset (sc+32, q+4),
        # Q6_K with (sc+128, q+32) and Q8_0 its codes as q+128, so their zero
        # blocks are not all-zero bytes; every format decodes to 0.
        if f not in ("Q3_K", "Q8_0", "Q6_K"):
            assert not p.any()
        u = orc.unpack(f, p, 3, 300)
        assert not u.any()


def _grid_weights(fmt, rng, rows, nb):
    """Weights that lie exactly on a format grid whose fields the quantizer
    must recover: largest sub-scale / sub-min at their maximum, every
    sub-block containing its extreme codes."""
    if fmt in ("Q2_K", "Q4_K"):
        L, S, sub = (3, 15, 16) if fmt == "Q2_K" else (15, 63, 32)
        d0, m0 = np.float32(2.0 ** -8), np.float32(2.0 ** -9)
        w = np.zeros((rows, nb * 256), np.float32)
        for r in range(rows):
            for b in range(nb):
                nsub = 256 // sub
                sc = rng.integers(1, S + 1, nsub); sc[0] = S
                m = rng.integers(0, S + 1, nsub); m[1] = S
                for j in range(nsub):
                    q = rng.integers(0, L + 1, sub); q[0] = 0; q[1] = L
                    w[r, b * 256 + j * sub: b * 256 + (j + 1) * sub] = d0 * sc[j] * q - m0 * m[j]
        return w
    if fmt == "Q3_K":
        d0 = np.float32(2.0 ** -8)
        w = np.zeros((rows, nb * 256), np.float32)
        for r in range(rows):
            for b in range(nb):
                sc = rng.integers(1, 32, 16) * rng.choice([-1, 1], 16); sc[0] = 31
                for j in range(16):
                    q = rng.integers(-3, 4, 16); q[2] = -4
                    w[r, b * 256 + j * 16: b * 256 + (j + 1) * 16] = d0 * sc[j] * q
        return w
    if fmt == "Q6_K":
        d0 = np.float32(2.0 ** -8)
        w = np.zeros((rows, nb * 256), np.float32)
        for r in range(rows):
            for b in range(nb):
                sc = rng.integers(1, 128, 16) * rng.choice([-1, 1], 16); sc[0] = 127
                for j in range(16):
                    q = rng.integers(-31, 32, 16); q[2] = -32
                    w[r, b * 256 + j * 16: b * 256 + (j + 1) * 16] = d0 * sc[j] * q
        return w
    if fmt == "BF16":
        # random bf16 values: the top 16 bits of random float32 values
        v = (rng.normal(0, 1, (rows, nb * 32)) * 2.0 ** rng.integers(-60, 60, (rows, nb * 32))).astype(np.float32)
        return (v.view(np.uint32) & np.uint32(0xFFFF0000)).view(np.float32)
    d0 = np.float32(2.0 ** -7)
    q = rng.integers(-127, 128, (rows, nb * 32)); q[:, ::32] = 127
    return (d0 * q).astype(np.float32)


@pytest.mark.parametrize("fmt", FMTS)
def test_grid_blocks_round_trip_exactly(orc, fmt):
    rng = np.random.default_rng(5)
    w = _grid_weights(fmt, rng, 3, 2)
    p = orc.pack(fmt, w)
    u = orc.unpack(fmt, p, *w.shape)
    np.testing.assert_array_equal(u, w)
    np.testing.assert_array_equal(orc.pack(fmt, u), p)


@pytest.mark.parametrize("fmt", ["Q2_K", "Q4_K", "Q3_K", "Q6_K"])
def test_codes_are_nearest_grid_points(orc, fmt):
    """Within a sub-block every dequantized value is one point of an
    arithmetic grid; the chosen point must be the nearest one to w that the
    code range allows (brute force over all codes of the grid)."""
    rng = np.random.default_rng(1)
    w = rng.normal(0, 0.02, (4, 512)).astype(np.float32)
    u = orc.unpack(fmt, orc.pack(fmt, w), 4, 512).astype(np.float64)
    sub = 32 if fmt == "Q4_K" else 16
    ncode = {"Q2_K": 4, "Q4_K": 16, "Q3_K": 8, "Q6_K": 64}[fmt]
    for r in range(4):
        for s in range(0, 512, sub):
            ws, us = w[r, s:s + sub].astype(np.float64), u[r, s:s + sub]
            levels = np.unique(us)
            if len(levels) < 2:
                continue
            step = np.min(np.diff(levels))
            # reconstruct the full grid of this sub-block from its smallest value
            if fmt in ("Q3_K", "Q6_K"):
                cand = [levels[0] + step * i for i in range(-ncode, 2 * ncode)]
            else:
                cand = [levels[0] + step * i for i in range(-ncode, ncode)]
            cand = np.array(cand)
            for wi, ui in zip(ws, us):
                best = np.min(np.abs(cand - wi))
                # chosen value is the nearest grid point (ties within rounding),
                # unless the nearest one lies outside the code range (clamped)
                assert abs(ui - wi) <= best + 1e-7 or ui in (levels[0], levels[-1])


@pytest.mark.parametrize("fmt", FMTS)
def test_error_within_closed_form_bound(orc, fmt):
    rng = np.random.default_rng(2)
    w = rng.normal(0, 0.02, (8, 768)).astype(np.float32)
    u = orc.unpack(fmt, orc.pack(fmt, w), *w.shape)
    err = np.abs(u.astype(np.float64) - w)
    if fmt == "Q8_0":
        blk = np.abs(w).reshape(8, -1, 32).max(-1, keepdims=True)
        bound = (blk / 127.0 * (0.5 + 2 ** -10) + 1e-9).repeat(32, -1).reshape(8, -1)
        assert (err <= bound).all()
        return
    if fmt == "BF16":
        # round to nearest bf16 (8 significant bits): half a unit in the last
        # place is at most 2^-8 of |w|
        assert (err <= np.abs(w.astype(np.float64)) * 2.0 ** -8).all()
        return
    if fmt == "Q6_K":
        ws = w.reshape(8, -1, 16, 16).astype(np.float64)
        step = np.abs(ws).max(-1) / 32.0                      # |scale_j|: the extreme weight maps to -32
        dmax = step.max(-1, keepdims=True) / 127 * (1 + 2 ** -10)
        # grid step g = d sc with |g - scale_j| <= d/2.  Unclamped codes miss
        # by <= g/2; a code clamped at +31 misses by <= |scale| + 15.5 d; one
        # clamped at -32 by <= 16 d.
        bound = np.repeat((step + 16.5 * dmax)[..., None], 16, -1).reshape(8, -1)
        assert (err <= bound + 1e-9).all(), float((err - bound).max())
        return
    L, S, sub = {"Q2_K": (3, 15, 16), "Q4_K": (15, 63, 32), "Q3_K": (4, 31, 16)}[fmt]
    ws = w.reshape(8, -1, 256 // sub, sub).astype(np.float64)
    if fmt == "Q3_K":
        step = np.abs(ws).max(-1) / 4.0                       # |scale_j|
        dmax = step.max(-1, keepdims=True) / S * (1 + 2 ** -10)
        # The grid holds codes -4..3 times the sub-scale, the extreme weight
        # mapping to -4: weights at the other end of the sub-block can clamp
        # at +3 steps, i.e. lose up to one whole step.  Plus the sub-scale
        # rounding: |d sc - scale| <= d/2 per code unit, |q-4| <= 4.
        bound = step + 4 * dmax / 2 + dmax * 0.5
    else:
        lo = np.minimum(0, ws.min(-1)); hi = ws.max(-1)
        step = (hi - lo) / L
        dmax = step.max(-1, keepdims=True) / S * (1 + 2 ** -10)
        mmax = (-lo).max(-1, keepdims=True) / S * (1 + 2 ** -10)
        bound = step / 2 + L * dmax / 2 + mmax / 2 + dmax
    bound = np.repeat(bound[..., None], sub, -1).reshape(8, -1)
    assert (err <= bound + 1e-9).all(), float((err - bound).max())


def test_pack_rejects_nonfinite(orc):
    w = np.zeros((1, 32), np.float32); w[0, 3] = np.nan
    with pytest.raises(ValueError):
        orc.pack("Q8_0", w)


def test_bf16_pack_rejects_values_beyond_its_range(orc):
    # the largest float32 rounds to bf16 infinity
    w = np.zeros((1, 32), np.float32); w[0, 5] = np.finfo(np.float32).max
    with pytest.raises(ValueError):
        orc.pack("BF16", w)
    w[0, 5] = np.float32(3.3895313892515355e38)        # largest bf16: kept
    assert orc.unpack("BF16", orc.pack("BF16", w), 1, 32)[0, 5] == w[0, 5]
