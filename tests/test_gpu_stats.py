"""Device expert histogram and pruning scores (arXiv 2509.25689 Sec. 3.1)
through the C ABI against the oracle (oracle/prune.py): counts and the
exact fixed-point weight sums bit for bit, f_e, s_e, I_e bit for bit, and
the kept set."""
import numpy as np
import pytest

from tests.gpu_helpers import mq_lib, tokens
from workloads.configs import LayerSpec

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def torch_cuda():
    import torch
    assert torch.cuda.is_available()
    return torch


def _oracle_all(idx, w, E, alpha, r):
    """Oracle counts, fixed-point sums, f, s, I and the kept ids."""
    from oracle import prune as R
    idx_l, w_l = np.asarray(idx).tolist(), np.asarray(w).tolist()
    count, fsum = R.expert_counts_and_sums(idx_l, w_l, E)
    T = len(idx_l)
    f = np.array([c / T if T > 0 else 0.0 for c in count])
    s = np.array([(fsum[e] / 2 ** 64) / count[e] if count[e] > 0 else 0.0 for e in range(E)])
    keep, scores = R.prune(idx_l, w_l, E, alpha, r)
    return count, fsum, f, s, np.array(scores), keep


def _device_stats(torch, batches, E, top_k, alpha, r):
    """Accumulate device batches [(idx_dev, w_dev, n_tokens)]; returns the raw
    buffer fields and the score outputs."""
    mq = mq_lib()
    nb = mq.mq_expert_stats_bytes(E)
    stats = torch.empty(nb, dtype=torch.uint8, device="cuda")
    mq.mq_expert_stats_reset(stats, E)
    for idx_d, w_d, n in batches:
        mq.mq_expert_stats_add(stats, E, idx_d, w_d, n, top_k)
    freq = torch.empty(E, dtype=torch.float64, device="cuda")
    mean_w = torch.empty(E, dtype=torch.float64, device="cuda")
    scores = torch.empty(E, dtype=torch.float64, device="cuda")
    keep = torch.full((E,), -1, dtype=torch.int32, device="cuda")
    k = mq.mq_expert_stats_scores(stats, E, alpha, r, freq, mean_w, scores, keep)
    torch.cuda.synchronize()
    raw = stats.cpu().numpy()
    n_tok = int(raw[0:8].view(np.uint64)[0])
    err = int(raw[8:12].view(np.uint32)[0])
    count = raw[16:16 + 8 * E].view(np.uint64)
    lo = raw[16 + 8 * E:16 + 16 * E].view(np.uint64)
    hi = raw[16 + 16 * E:16 + 24 * E].view(np.int64)
    fsum = [int(hi[e]) * 2 ** 64 + int(lo[e]) for e in range(E)]
    return dict(n_tokens=n_tok, err=err, count=count.astype(np.int64), fsum=fsum, freq=freq.cpu().numpy(),
                mean_w=mean_w.cpu().numpy(), scores=scores.cpu().numpy(), keep=keep.cpu().numpy()[:k], k=k)


def _check(dev, ref):
    count, fsum, f, s, scores, keep = ref
    np.testing.assert_array_equal(dev["count"], np.array(count, np.int64))
    assert dev["fsum"] == fsum
    np.testing.assert_array_equal(dev["freq"].view(np.uint64), f.view(np.uint64))
    np.testing.assert_array_equal(dev["mean_w"].view(np.uint64), s.view(np.uint64))
    np.testing.assert_array_equal(dev["scores"].view(np.uint64), scores.view(np.uint64))
    assert list(dev["keep"]) == keep


def test_stats_from_device_routing_match_oracle(torch_cuda, orc):
    """A calibration stream routed on the GPU by the unpruned V3 router (256
    experts, 8 groups, top-8) in four batches of different sizes, the
    histogram fed straight from the router's device outputs."""
    mq = mq_lib()
    from workloads.synth import draw_router
    spec = LayerSpec(name="v3_unpruned_router", hidden=7168, inter=2048, n_experts=256, n_groups=8, topk_group=4,
                     top_k=8, tokens=1536, has_shared=True, router_std=1 / 7168 ** 0.5, bias_std=0.01)
    rw, b = draw_router(spec, 4)
    cfg = mq.make_cfg(spec.hidden, spec.inter, 256, 8, 4, 8, spec.routed_scale, True)
    router_w, bias = torch_cuda.from_numpy(rw).cuda(), torch_cuda.from_numpy(b).cuda()
    batches, host_x = [], []
    for bi, T in enumerate((1, 7, 512, 1016)):
        x = tokens(spec, 40 + bi, T)
        host_x.append(x)
        xd = torch_cuda.from_numpy(np.ascontiguousarray(x).view(np.int16)).cuda()
        idx = torch_cuda.empty((T, 8), dtype=torch_cuda.int32, device="cuda")
        w = torch_cuda.empty((T, 8), dtype=torch_cuda.float32, device="cuda")
        wsb = mq.moe_quant_workspace_size(cfg, T)
        ws = torch_cuda.empty(wsb, dtype=torch_cuda.uint8, device="cuda")
        mq.moe_quant_route(cfg, T, xd, router_w, bias, idx, w, workspace=ws, ws_bytes=wsb)
        batches.append((idx, w, T, ws))
    dev = _device_stats(torch_cuda, [(i, w, T) for i, w, T, _ in batches], 256, 8, 0.5, 0.75)
    # the oracle routes the same tokens itself
    layer = orc.make_layer(spec.hidden, spec.inter, 256, 8, 4, 8, spec.routed_scale, True)
    ridx, rwt = [], []
    for x in host_x:
        a, bw, _, _ = orc.route(layer, x, rw, b)
        ridx.append(a)
        rwt.append(bw)
    ridx, rwt = np.concatenate(ridx), np.concatenate(rwt)
    assert dev["n_tokens"] == 1536 and dev["err"] == 0 and dev["k"] == 192
    _check(dev, _oracle_all(ridx, rwt, 256, 0.5, 0.75))
    # and the library's host routine on the same stream gives the same bits
    keep_h, scores_h = mq.mq_expert_importance(ridx, rwt, 256, 0.5, 0.75)
    np.testing.assert_array_equal(scores_h.view(np.uint64), dev["scores"].view(np.uint64))


@pytest.mark.parametrize("alpha,r", [(0.5, 0.75), (0.0, 0.5), (1.0, 0.3), (0.25, 1.0)])
def test_stats_hard_weights(torch_cuda, alpha, r):
    """Weights spread over 2^-80 .. 2^31 (below 2^-40 they round to 2^-64
    units), negative ones, a stream a running sum gets wrong, zipf-skewed
    ids, split into uneven batches: every field bit-exact."""
    rng = np.random.default_rng(7)
    E, K, T = 96, 6, 3000
    p = rng.zipf(1.3, E).astype(np.float64)
    p /= p.sum()
    idx = np.stack([rng.choice(E, K, replace=False, p=p) for _ in range(T)]).astype(np.int32)
    w = (rng.random((T, K)) * 2.0 ** rng.integers(-80, 31, (T, K))).astype(np.float32)
    w[rng.random((T, K)) < 0.1] *= -1
    w[:300, 0] = np.float32(2.0 ** -60)
    idx[:300, 0] = 5
    idx[300, :] = np.arange(K)
    w[300, 0] = np.float32(1.0)
    w[rng.random((T, K)) < 0.02] = 0.0
    ref = _oracle_all(idx, w, E, alpha, r)
    cuts = [0, 1, 2, 1000, 1001, 2999, T]
    batches = []
    for a, bnd in zip(cuts[:-1], cuts[1:]):
        batches.append((torch_cuda.from_numpy(idx[a:bnd].copy()).cuda(), torch_cuda.from_numpy(w[a:bnd].copy()).cuda(),
                        bnd - a))
    dev = _device_stats(torch_cuda, batches, E, K, alpha, r)
    assert dev["n_tokens"] == T and dev["err"] == 0
    _check(dev, ref)


def test_stats_large_stream_many_ctas(torch_cuda):
    """A stream large enough for every CTA of the grid to flush a partial
    histogram (262,144 tokens x top-8 over 256 experts, zipf ids)."""
    rng = np.random.default_rng(11)
    E, K, T = 256, 8, 262144
    ranks = np.minimum(rng.zipf(1.1, (T, K)) - 1, E - 1)
    idx = ((ranks * 37 + 11) % E).astype(np.int32)            # repeats within a row are allowed here
    w = (rng.random((T, K)) * 2.5).astype(np.float32)
    dev = _device_stats(torch_cuda, [(torch_cuda.from_numpy(idx).cuda(), torch_cuda.from_numpy(w).cuda(), T)], E, K,
                        0.5, 0.75)
    np.testing.assert_array_equal(dev["count"], np.bincount(idx.reshape(-1), minlength=E))
    _check(dev, _oracle_all(idx, w, E, 0.5, 0.75))


def test_stats_skip_bad_entries(torch_cuda):
    """Ids outside 0..E-1 and non-finite or too large weights are skipped and
    flagged (bits 1 and 2); the rest is accumulated as usual."""
    E, K = 8, 2
    idx = np.array([[0, 1], [8, 2], [-1, 3], [4, 5], [6, 7]], np.int32)
    w = np.array([[0.5, 0.25], [1.0, np.inf], [1.0, 0.125], [np.nan, 2.0 ** 32], [0.75, -0.5]], np.float32)
    dev = _device_stats(torch_cuda, [(torch_cuda.from_numpy(idx).cuda(), torch_cuda.from_numpy(w).cuda(), 5)], E, K,
                        0.5, 0.5)
    assert dev["err"] == 3 and dev["n_tokens"] == 5
    assert list(dev["count"]) == [1, 1, 0, 1, 0, 0, 1, 1]
    assert dev["fsum"] == [2 ** 63, 2 ** 62, 0, 2 ** 61, 0, 0, 3 * 2 ** 62, -(2 ** 63)]
    # the first bad flag alone
    dev = _device_stats(torch_cuda, [(torch_cuda.from_numpy(idx[1:3]).cuda(),
                                      torch_cuda.from_numpy(np.ones((2, 2), np.float32)).cuda(), 2)], E, K, 0.5, 0.5)
    assert dev["err"] == 1


def test_stats_empty_stream(torch_cuda):
    dev = _device_stats(torch_cuda, [], 16, 4, 0.5, 0.75)
    assert dev["n_tokens"] == 0 and dev["err"] == 0 and dev["k"] == 12
    assert (dev["scores"] == 0).all() and list(dev["keep"]) == list(range(12))


def test_stats_max_experts(torch_cuda):
    rng = np.random.default_rng(3)
    E, K, T = 1024, 8, 4096
    idx = np.stack([rng.choice(E, K, replace=False) for _ in range(T)]).astype(np.int32)
    w = rng.random((T, K)).astype(np.float32)
    dev = _device_stats(torch_cuda, [(torch_cuda.from_numpy(idx).cuda(), torch_cuda.from_numpy(w).cuda(), T)], E, K,
                        0.5, 0.75)
    _check(dev, _oracle_all(idx, w, E, 0.5, 0.75))
