"""Checkpoint of a packed layer (raw planar streams + JSON header): round
trip, and corrupted or truncated files refused before anything reaches the
kernels.  CPU only."""
import json
import os

import numpy as np
import pytest


@pytest.fixture(scope="module")
def mq():
    import paper_2509_25689_gb300 as m
    return m


def _layer(mq, rng, E=4, H=256, I=128, shared=True):
    fm = rng.integers(1, 5, size=(E + shared, 3)).astype(np.uint8)
    pk = lambda f, r, c: mq.mq_pack(int(f), rng.normal(0, 0.02, (r, c)).astype(np.float32))
    trips = [(pk(fm[e, 0], I, H), pk(fm[e, 1], I, H), pk(fm[e, 2], H, I)) for e in range(E + shared)]
    cfg = dict(hidden=H, inter=I, n_experts=E, n_groups=2, topk_group=1, top_k=2, routed_scale=2.5,
               has_shared=int(shared))
    rw = rng.normal(0, 0.06, (E, H)).astype(np.float32)
    b = rng.normal(0, 0.01, E).astype(np.float32)
    return cfg, fm, trips[:E], (trips[E] if shared else None), rw, b


def test_round_trip(mq, tmp_path):
    from paper_2509_25689_gb300.checkpoint import load_layer, save_layer
    cfg, fm, ex, sh, rw, b = _layer(mq, np.random.default_rng(0))
    save_layer(str(tmp_path), cfg, fm, ex, sh, rw, b)
    got = load_layer(str(tmp_path))
    assert got["cfg"] == cfg
    np.testing.assert_array_equal(got["formats"], fm)
    np.testing.assert_array_equal(got["router_w"], rw)
    np.testing.assert_array_equal(got["bias"], b)
    for a, c in zip(got["experts"] + [got["shared"]], ex + [sh]):
        for j in range(3):
            np.testing.assert_array_equal(a[j], c[j])
    hdr = json.load(open(tmp_path / "layer.json"))
    assert all(s["offset"] % 256 == 0 for s in hdr["streams"])


def test_no_shared_expert_and_no_bias(mq, tmp_path):
    from paper_2509_25689_gb300.checkpoint import load_layer, save_layer
    cfg, fm, ex, sh, rw, _ = _layer(mq, np.random.default_rng(1), shared=False)
    save_layer(str(tmp_path), cfg, fm, ex, None, rw, None)
    got = load_layer(str(tmp_path))
    assert got["shared"] is None and got["bias"] is None
    np.testing.assert_array_equal(got["experts"][3][2], ex[3][2])


def test_corruption_and_truncation_are_refused(mq, tmp_path):
    from paper_2509_25689_gb300.checkpoint import load_layer, save_layer
    cfg, fm, ex, sh, rw, b = _layer(mq, np.random.default_rng(2))
    save_layer(str(tmp_path), cfg, fm, ex, sh, rw, b)
    blob = bytearray(open(tmp_path / "layer.bin", "rb").read())
    hdr = json.load(open(tmp_path / "layer.json"))
    s = hdr["streams"][5]
    blob[s["offset"] + 3] ^= 0x40
    open(tmp_path / "layer.bin", "wb").write(bytes(blob))
    with pytest.raises(ValueError, match="checksum"):
        load_layer(str(tmp_path))
    blob[s["offset"] + 3] ^= 0x40
    open(tmp_path / "layer.bin", "wb").write(bytes(blob[:-100]))
    with pytest.raises(ValueError, match="truncated"):
        load_layer(str(tmp_path))
    # a header whose format no longer matches the stream's size
    open(tmp_path / "layer.bin", "wb").write(bytes(blob))
    hdr["formats"][0][0] = 4 if hdr["formats"][0][0] != 4 else 1
    json.dump(hdr, open(tmp_path / "layer.json", "w"))
    with pytest.raises(ValueError, match="needs"):
        load_layer(str(tmp_path))


def test_save_checks_sizes_against_the_formats(mq, tmp_path):
    from paper_2509_25689_gb300.checkpoint import save_layer
    cfg, fm, ex, sh, rw, b = _layer(mq, np.random.default_rng(3))
    bad = list(ex)
    bad[1] = (bad[1][0][:-16], bad[1][1], bad[1][2])
    with pytest.raises(ValueError, match="needs"):
        save_layer(str(tmp_path), cfg, fm, bad, sh, rw, b)
    with pytest.raises(ValueError):
        save_layer(str(tmp_path), cfg, fm, ex, None, rw, b)   # has_shared but no shared expert


@pytest.mark.parametrize("edit,match", [
    (lambda h: h["formats"].pop(), "formats: shape"),                       # one row short
    (lambda h: h["formats"][1].__setitem__(2, 9), "unknown format"),          # bad code
    (lambda h: h["cfg"].__setitem__("n_groups", 3), "n_groups"),              # does not divide E
    (lambda h: h["cfg"].__setitem__("top_k", 64), "top_k"),
    (lambda h: h["cfg"].__setitem__("hidden", 200), "hidden"),
    (lambda h: h["cfg"].pop("inter"), "missing"),
])
def test_inconsistent_headers_are_refused(mq, tmp_path, edit, match):
    from paper_2509_25689_gb300.checkpoint import load_layer, save_layer
    cfg, fm, ex, sh, rw, b = _layer(mq, np.random.default_rng(4))
    save_layer(str(tmp_path), cfg, fm, ex, sh, rw, b)
    hdr = json.load(open(tmp_path / "layer.json"))
    edit(hdr)
    json.dump(hdr, open(tmp_path / "layer.json", "w"))
    with pytest.raises(ValueError, match=match):
        load_layer(str(tmp_path))


def test_bias_of_the_wrong_length_is_refused(mq, tmp_path):
    from paper_2509_25689_gb300.checkpoint import load_layer, save_layer
    cfg, fm, ex, sh, rw, b = _layer(mq, np.random.default_rng(5))
    save_layer(str(tmp_path), cfg, fm, ex, sh, rw, b)
    hdr = json.load(open(tmp_path / "layer.json"))
    streams = {s["name"]: s for s in hdr["streams"]}
    # the header's bias entry points at the router's bytes (checksum intact)
    streams["bias"].update({k: streams["router_w"][k] for k in ("offset", "bytes", "sha256")})
    json.dump(hdr, open(tmp_path / "layer.json", "w"))
    with pytest.raises(ValueError, match="bias"):
        load_layer(str(tmp_path))
