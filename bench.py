"""Benchmark: quantized MoE layer decode on GB300.

One step = one pass of the whole layer (router logits, group-limited top-k,
permutation, SwiGLU gate/up, down + weighted combine + shared expert) over
one batch of synthetic tokens, through the C ABI (moe_quant_forward).
Default workload: one DeepSeek-V3-shaped layer (hidden 7168, expert
intermediate 2048, 192 surviving experts of 256, 8 groups / 4 kept, top-8,
shared expert), decode batch of 1 token, gate/up Q2_K-style, down
Q3_K-style, shared expert Q8_0.  Packed weights are drawn on the device;
every step gets a fresh token and the L2 is flushed (256 MB write) before it.

  python bench.py [--gpus N] [--steps K] [--warmup W] [--impl native|reference]

With N > 1 (torchrun, one rank per GPU) every rank runs an independent
replica of the layer (weak scaling; no collective on the data path).
"""
from __future__ import annotations

import argparse
import json
import math
import os
import statistics
import subprocess
import sys
import tempfile
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "tokens/s and achieved HBM GB/s (% of peak) for quantized MoE layer decode, 1 GB300"
WORKLOAD = "v3_decode_t1"
FLUSH_BYTES = 256 << 20


def _peaks():
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            p = json.load(f)
        return float(p["hbm_gbs"]), "measured"
    except Exception:
        return 6800.0, "fallback"


# DRAM traffic per launch of the decode FFN kernels, from the committed ncu
# summary; reported only for the captured workload and only while the kernel
# sources are the ones captured.
PROFILE_SUMMARY = os.path.join(ROOT, "profiles", "ffn_kernel_v3_decode_t1.md")
PROFILE_WORKLOAD = "v3_decode_t1"
KERNEL_SOURCES = ("k_decode.cu", "mq_actprep.cuh", "mq_layout.h", "mq_internal.h")


def _profiled_traffic(kernel: str, workload: str = PROFILE_WORKLOAD):
    if workload != PROFILE_WORKLOAD:
        return None
    import hashlib
    try:
        text = open(PROFILE_SUMMARY).read()
        h = hashlib.sha256()
        for f in KERNEL_SOURCES:
            with open(os.path.join(ROOT, "paper_2509_25689_gb300", "csrc", f), "rb") as fh:
                h.update(fh.read())
        fields = dict(line.split(": ", 1) for line in text.splitlines() if ": " in line and " " not in line.split(": ")[0])
        if fields.get("kernel_sources_sha256_16", "").strip() != h.hexdigest()[:16]:
            return None
        key = {"ffn_mma": "dram_bytes_per_launch_ffn"}.get(kernel)
        return int(fields[key]) if key in fields else None
    except Exception:
        return None


class ClockSampler:
    """nvidia-smi clocks/throttle sampling during the timed region."""

    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index: int):
        self.gpu = gpu_index
        self.proc = None
        self.path = None

    def start(self):
        fd, self.path = tempfile.mkstemp(suffix=".csv")
        os.close(fd)
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--id={self.gpu}", f"--query-gpu={self.FIELDS}", "--format=csv,noheader,nounits",
                 "-lms", "100", "-f", self.path], stdout=subprocess.DEVNULL, stderr=subprocess.DEVNULL)
        except Exception:
            self.proc = None
        time.sleep(0.3)

    def stop(self):
        if self.proc is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        time.sleep(0.25)
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except Exception:
            self.proc.kill()
        sm, smax, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        with open(self.path) as f:
            for line in f:
                c = [s.strip() for s in line.split(",")]
                if len(c) < 9:
                    continue
                try:
                    sm.append(float(c[1])); smax.append(float(c[2]))
                except ValueError:
                    continue
                for n, v in zip(names, c[5:9]):
                    if v.lower().startswith("active"):
                        reasons.add(n)
        os.unlink(self.path)
        return {"sm_mhz": statistics.median(sm) if sm else None, "sm_max_mhz": max(smax) if smax else None,
                "reasons": sorted(reasons), "samples": len(sm)}


def step_bytes(spec, fmts, idx_steps):
    """Algorithmic bytes per step for each kernel (packed bytes of the tensors
    each kernel must read, plus activations)."""
    from workloads.configs import packed_bytes
    H, I, E, T, K = spec.hidden, spec.inter, spec.n_experts, spec.tokens, spec.top_k
    gu = lambda e: packed_bytes(int(fmts[e, 0]), I, H) + packed_bytes(int(fmts[e, 1]), I, H)
    dn = lambda e: packed_bytes(int(fmts[e, 2]), H, I)
    sh = E if spec.has_shared else None
    out = []
    for idx in idx_steps:
        touched = sorted(set(int(e) for e in idx.reshape(-1)))
        b_gu = sum(gu(e) for e in touched) + (gu(sh) if sh is not None else 0) + T * H * 2 + (T * K + T) * I * 4
        b_dn = sum(dn(e) for e in touched) + (dn(sh) if sh is not None else 0) + (T * K + T) * I * 4 + T * H * 4
        b_rt = E * H * 4 + T * H * 2 + T * E * 4
        quant = sum(gu(e) + dn(e) for e in touched) + ((gu(sh) + dn(sh)) if sh is not None else 0)
        out.append({"ffn_mma": b_gu + b_dn, "gateup_mma": b_gu, "down_mma": b_dn, "router_logits": b_rt,
                    "quantized": quant,
                    "total": b_gu + b_dn + b_rt, "gateup_tc": b_gu, "down_tc": b_dn,
                    "gateup_tgemv": b_gu, "down_tgemv": b_dn})
    return out


def flops_active_per_token(k_layers, P, has_shared):
    """FLOPs_active = 2 sum_i k_i P_i per token over the layers (Sec. 3.2;
    P = parameters of one routed expert), and the same with each layer's
    shared expert (always active) added."""
    routed = 2 * sum(int(k) for k in k_layers) * P
    return {"routed": routed, "with_shared": routed + (2 * len(k_layers) * P if has_shared else 0)}


def step_flops(spec):
    """Dense-contraction FLOPs per step of the expert FFN kernels: every routed
    assignment and every shared-expert row does gate and up (2 x 2 H I) and
    down (2 H I)."""
    rows = spec.tokens * spec.top_k + (spec.tokens if spec.has_shared else 0)
    hi = spec.hidden * spec.inter
    return {"gateup_tc": rows * 4 * hi, "down_tc": rows * 2 * hi}


def _tensor_peak():
    """Dense fp16 tensor peak: the measured bf16 figure (fp16 and bf16 have the
    same nominal dense rate, 2.25 PFLOP/s)."""
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            p = json.load(f)
        return float(p["bf16_tflops"]), "measured bf16 burst (fp16 nominal ratio 1.0)"
    except Exception:
        return 1900.0, "fallback"


def cpu_baseline(host_layer, x_full, budget_s=12.0, sample_tokens=8, openmp=False):
    """The oracle as it stands (plain C, fp64 FFN) timed on the host cores on
    a bounded sample of the workload, scaled to the whole workload.

    The oracle unpacks every expert a call touches once and then applies it
    to that expert's tokens, so its cost per call is (distinct experts) x
    unpack + (assignments) x apply.  A sample of at most `sample_tokens` of
    the workload's tokens is timed end to end, the unpack of the sample's
    experts is timed on its own, and the two per-unit costs are scaled to the
    full batch's own counts (its distinct experts from an untimed oracle
    routing of every token, its assignments T * k + T).  For one-token
    workloads the sample is the workload.  openmp: the oracle's OpenMP build
    on all host cores (identical results)."""
    import oracle
    oracle.build()
    oracle.use_openmp(openmp)
    try:
        spec = host_layer.spec
        T = x_full.shape[0]
        n_s = min(T, sample_tokens)
        t_fwd, t_unpack, d_s, a_s, done = 0.0, 0.0, 0, 0, 0
        for i in range(0, T, n_s):
            xs = x_full[i:i + n_s]
            tf, tu, ds = host_layer.timed_parts(oracle, xs)
            t_fwd += tf
            t_unpack += tu
            d_s += ds
            a_s += xs.shape[0] * spec.top_k + (xs.shape[0] if spec.has_shared else 0)
            done += xs.shape[0]
            if t_fwd + t_unpack > budget_s or n_s == T:
                break
        if done == T:
            value = T / t_fwd
            how = f"all {T} token(s) of the workload, {t_fwd:.1f} s"
        else:
            d_full = host_layer.distinct_experts(oracle, x_full)
            a_full = T * spec.top_k + (T if spec.has_shared else 0)
            per_expert = t_unpack / d_s
            per_assign = max(t_fwd - t_unpack, 0.0) / a_s
            t_full = d_full * per_expert + a_full * per_assign
            value = T / t_full
            how = (f"{done} of the workload's {T} tokens timed ({t_fwd:.1f} s, {d_s} expert unpacks in "
                   f"{t_unpack:.1f} s); scaled to its {d_full} distinct experts and {a_full} assignments")
        cores = os.cpu_count() if openmp else 1
        return {"value": value, "unit": "tokens/s", "cores": cores, "kind": "oracle",
                "build": "OpenMP, all host cores" if openmp else "single thread",
                "sample": f"{spec.name}: {how}"}
    finally:
        oracle.use_openmp(False)


class HostOracleLayer:
    """Host-only layer for the oracle: same seeded recipe as the device layer;
    packed tensors are drawn on the host for the experts a token touches."""

    def __init__(self, spec, seed):
        from workloads.synth import draw_formats, draw_router
        self.spec, self.seed = spec, seed
        self.fmts = draw_formats(spec, seed)
        self.router_w, self.bias = draw_router(spec, seed)
        self.cache = {}

    def _layer(self, orc):
        spec = self.spec
        return orc.make_layer(spec.hidden, spec.inter, spec.n_experts, spec.n_groups, spec.topk_group,
                              spec.top_k, spec.routed_scale, spec.has_shared)

    def distinct_experts(self, orc, x_bits):
        """Experts one oracle call on x_bits unpacks (routed ones plus the shared one)."""
        idx, _, _, _ = orc.route(self._layer(orc), x_bits, self.router_w, self.bias)
        return len(set(int(e) for e in idx.reshape(-1))) + (1 if self.spec.has_shared else 0)

    def timed_parts(self, orc, x_bits):
        """(time of one oracle call on x_bits, time of unpacking its experts
        alone, number of those experts)."""
        from workloads.synth import draw_packed_layer_host, tensor_shapes
        spec = self.spec
        layer = self._layer(orc)
        idx, _, _, _ = orc.route(layer, x_bits, self.router_w, self.bias)
        n = spec.n_experts + (1 if spec.has_shared else 0)
        used = set(int(e) for e in idx.reshape(-1)) | set(range(spec.n_experts, n))
        for e in used:
            if e not in self.cache:
                self.cache[e] = draw_packed_layer_host(spec, self.seed, self.fmts, experts=[e])[e]
        dummy = np.zeros(16, np.uint8)
        g = [self.cache[e][0] if e in used else dummy for e in range(n)]
        u = [self.cache[e][1] if e in used else dummy for e in range(n)]
        d = [self.cache[e][2] if e in used else dummy for e in range(n)]
        t0 = time.perf_counter()
        orc.moe_forward(layer, x_bits, self.router_w, self.bias, g, u, d, self.fmts)
        t_fwd = time.perf_counter() - t0
        shapes = tensor_shapes(spec)
        t0 = time.perf_counter()
        for e in used:
            for j in range(3):
                orc.unpack(int(self.fmts[e, j]), self.cache[e][j], *shapes[j])
        t_unpack = time.perf_counter() - t0
        return t_fwd, t_unpack, len(used)

    def timed_forward(self, orc, x_bits):
        return self.timed_parts(orc, x_bits)[0]


class BenchLayer:
    def __init__(self, spec, seed):
        import torch
        import paper_2509_25689_gb300 as mq
        from workloads.synth import draw_formats, draw_router, random_packed_device, tensor_shapes
        self.mq, self.spec = mq, spec
        self.fmts = draw_formats(spec, seed)
        gen = torch.Generator(device="cuda")
        gen.manual_seed(seed * 7919 + 13)
        shapes = tensor_shapes(spec)
        n = spec.n_experts + (1 if spec.has_shared else 0)
        self.tensors = [tuple(random_packed_device(int(self.fmts[e, j]), *shapes[j], gen, "cuda") for j in range(3))
                        for e in range(n)]
        self.table = mq.ExpertTable(self.tensors[:spec.n_experts],
                                    self.tensors[spec.n_experts] if spec.has_shared else None)
        rw, b = draw_router(spec, seed)
        self.router_w_host, self.bias_host = rw, b
        self.router_w, self.bias = torch.from_numpy(rw).cuda(), torch.from_numpy(b).cuda()
        self.cfg = mq.make_cfg(spec.hidden, spec.inter, spec.n_experts, spec.n_groups, spec.topk_group,
                               spec.top_k, spec.routed_scale, spec.has_shared)
        self.wsb = mq.moe_quant_workspace_size(self.cfg, spec.tokens)
        self.ws = torch.empty(self.wsb, dtype=torch.uint8, device="cuda")
        self.out = torch.empty((spec.tokens, spec.hidden), dtype=torch.float32, device="cuda")
        self.wts = torch.empty((spec.tokens, spec.top_k), dtype=torch.float32, device="cuda")

    def forward(self, x, idx_out, out=None):
        self.mq.moe_quant_forward(self.cfg, self.spec.tokens, x, self.router_w, self.bias, self.table, self.fmts,
                                  self.out if out is None else out, idx_out, self.wts, self.ws, self.wsb)


def max_over_ranks(x: float, world: int, device) -> float:
    """Largest value of x over the ranks (the slowest rank's time)."""
    if world == 1:
        return float(x)
    import torch
    import torch.distributed as dist
    t = torch.tensor([float(x)], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def job_throughput(world: int, tokens_per_step: int, steps: int, ms_max: float) -> float:
    """Whole-job tokens/s: every rank's tokens over the slowest rank's time."""
    return world * tokens_per_step * steps / (ms_max / 1e3)


def measure_layer(spec, K, W, rank=0, world=1, local=0):
    """One layer workload: K timed steps after W warm-up steps (L2 flushed
    before each), per-kernel times, end-to-end through host buffers.  Returns
    (result dict for rank 0 or None, the timed steps' token batches, the
    timed steps' expert ids)."""
    import torch
    import torch.distributed as dist
    from workloads.synth import draw_tokens

    T = spec.tokens
    layer = BenchLayer(spec, seed=rank)
    steps = W + K
    # a fresh token batch per step (decode); prefill cycles through a pool of
    # distinct batches of at most ~64 MB in total
    n_pool = min(steps, max(1, (64 << 20) // (T * spec.hidden * 2)))
    x_host = np.stack([draw_tokens(1000 + rank * 100003 + i, T, spec.hidden) for i in range(n_pool)])
    x_dev = torch.from_numpy(x_host.view(np.int16)).cuda()
    idx_all = torch.empty((steps, T, spec.top_k), dtype=torch.int32, device="cuda")
    xi = lambda i: i % n_pool
    flush = torch.empty(FLUSH_BYTES // 4, dtype=torch.int32, device="cuda")

    def barrier():
        torch.cuda.synchronize()
        if world > 1:
            dist.barrier()
        torch.cuda.synchronize()

    for i in range(W):
        flush.fill_(i)
        layer.forward(x_dev[xi(i)], idx_all[i])
    barrier()

    clocks = ClockSampler(local)
    clocks.start()
    evs = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(K)]
    barrier()
    t_wall0 = time.perf_counter()
    for i in range(K):
        flush.fill_(i)
        evs[i][0].record()
        layer.forward(x_dev[xi(W + i)], idx_all[W + i])
        evs[i][1].record()
    barrier()
    t_wall = time.perf_counter() - t_wall0
    clk = clocks.stop()
    # Per-kernel durations: the same K steps once more with a CUDA event pair
    # around every kernel on the launching stream (kept out of the timed
    # region above, where the events would add gaps between the kernels).
    layer.mq.mq_profile_enable(K * 8)
    for i in range(K):
        flush.fill_(i)
        layer.forward(x_dev[xi(W + i)], idx_all[W + i])
    barrier()
    kstats = layer.mq.mq_profile_collect()
    dev_ms = sum(a.elapsed_time(b) for a, b in evs)
    dev_ms_max = max_over_ranks(dev_ms, world, "cuda")

    # e2e through the C ABI with host buffers (pinned), copies inside the region
    x_pin = torch.from_numpy(x_host.view(np.int16)).pin_memory()
    out_pin = torch.empty((2, T, spec.hidden), dtype=torch.float32).pin_memory()   # ring of two
    x_step = torch.empty((T, spec.hidden), dtype=torch.int16, device="cuda")
    e2e_evs = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(K)]
    barrier()
    for i in range(K):
        flush.fill_(i)
        e2e_evs[i][0].record()
        x_step.copy_(x_pin[xi(W + i)], non_blocking=True)
        layer.forward(x_step, idx_all[W + i])
        out_pin[i % 2].copy_(layer.out, non_blocking=True)
        e2e_evs[i][1].record()
    barrier()
    e2e_ms = sum(a.elapsed_time(b) for a, b in e2e_evs)
    e2e_ms_max = max_over_ranks(e2e_ms, world, "cuda")

    idx_host = idx_all[W:].cpu().numpy()
    sb = step_bytes(spec, layer.fmts, idx_host)
    peak, peak_src = _peaks()
    quant_bytes = sum(s["quantized"] for s in sb)
    gbs = quant_bytes / (dev_ms / 1e3) / 1e9
    result = None
    if rank == 0:
        dominant = max(kstats, key=lambda s: s[2]) if kstats else None
        roof = None
        if dominant and dominant[0].endswith("_tc"):
            # prefill: the grouped GEMM is a dense contraction -> tensor roofline
            name, launches, tot_ms = dominant
            fl = step_flops(spec)[name]
            avg_s = tot_ms / launches / 1e3
            tpeak, tsrc = _tensor_peak()
            achieved = fl / avg_s / 1e12
            roof = {"bound": "tensor", "kernel": name, "achieved": round(achieved, 1), "peak": tpeak,
                    "unit": "TFLOP/s", "frac": round(achieved / tpeak, 4), "traffic": None, "peak_source": tsrc,
                    "algorithmic_flops_per_launch": int(fl), "avg_launch_us": round(avg_s * 1e6, 2)}
            dominant = None
        if dominant:
            name, launches, tot_ms = dominant
            per_launch_bytes = sum(s.get(name, 0) for s in sb) / max(len(sb), 1)
            avg_s = tot_ms / launches / 1e3
            achieved = per_launch_bytes / avg_s / 1e9
            roof = {"bound": "hbm", "kernel": name, "achieved": round(achieved, 1), "peak": peak, "unit": "GB/s",
                    "frac": round(achieved / peak, 4), "traffic": _profiled_traffic(name, spec.name), "peak_source": peak_src,
                    "algorithmic_bytes_per_launch": int(per_launch_bytes), "avg_launch_us": round(avg_s * 1e6, 2)}
        result = {
            "metric": METRIC, "value": round(job_throughput(world, T, K, dev_ms_max), 2), "unit": "tokens/s",
            "n_gpus": world, "steps": K, "warmup": W, "ms_per_step": round(dev_ms_max / K, 5),
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f16xf16->f32",
            "data": "synthetic (seeded random packed weights on device; fresh N(0,1) bf16 token per step)",
            "config": {"workload": f"{spec.name}: V3 MoE layer, hidden {spec.hidden}, inter {spec.inter}, "
                                   f"{spec.n_experts} experts + shared, G={spec.n_groups}/{spec.topk_group}, "
                                   f"top-{spec.top_k}, T={T}", "l2": "flushed (256 MB write) before every step",
                       "parallelism": f"replicas x{world}"},
            "flops_active_per_token": flops_active_per_token([spec.top_k], spec.expert_param_count(),
                                                             spec.has_shared),
            "achieved_hbm_gbs": round(gbs, 1), "hbm_frac_of_measured": round(gbs / peak, 4),
            "hbm_frac_of_8tbs": round(gbs / 8000.0, 4), "quantized_bytes_per_step": int(quant_bytes / K),
            "roofline": roof,
            "kernels": [{"name": n, "launches": l, "total_ms": round(ms, 4)} for n, l, ms in kstats],
            "gpu_launches": int(sum(l for _, l, _ in kstats)),
            "wall_s_timed_region": round(t_wall, 4),
            "clocks": clk,
            "e2e": {"value": round(job_throughput(world, T, K, e2e_ms_max), 2), "unit": "tokens/s",
                    "h2d_bytes_per_step": int(T * spec.hidden * 2), "d2h_bytes_per_step": int(T * spec.hidden * 4)},
        }
    del layer, x_dev, flush
    torch.cuda.empty_cache()
    return result, x_host[xi(W)], idx_host


def zipf_histogram(spec, idx_host):
    """Routed count histogram of a Zipf-skewed workload against its
    water-filled Zipf target (per expert), as reported beside the line."""
    from workloads.synth import zipf_ranks, zipf_target_counts
    T, E, K = spec.tokens, spec.n_experts, spec.top_k
    steps = idx_host.size // (T * K)
    counts = np.bincount(idx_host.reshape(-1), minlength=E) / max(steps, 1)
    target = zipf_target_counts(E, T * K, float(spec.zipf_s), T)[zipf_ranks(spec, 0)]
    return {"zipf_s": spec.zipf_s, "l1_distance_to_target": round(float(np.abs(counts - target).sum() / (T * K)), 4),
            "experts_touched": int((counts > 0).sum()), "top_count": float(counts.max()),
            "top_count_target": float(target.max())}


SUB_RECORDS = (("v3_decode_t32_mixed", 50, 5), ("v3_prefill_t2048_zipf", 10, 3))


def run_native(args):
    import torch
    import torch.distributed as dist
    from workloads import get_config

    rank = int(os.environ.get("RANK", "0"))
    world = int(os.environ.get("WORLD_SIZE", "1"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    torch.cuda.set_device(local)
    if world > 1:
        dist.init_process_group("nccl")
    spec = get_config(args.config)
    result, x_first, idx_host = measure_layer(spec, args.steps, args.warmup, rank, world, local)
    if result is not None and spec.zipf_s is not None:
        result["routing_histogram"] = zipf_histogram(spec, idx_host)
    if result is not None and world == 1 and not args.no_cpu_baseline:
        host = HostOracleLayer(spec, seed=0)
        result["cpu_baseline"] = cpu_baseline(host, x_first, openmp=True)
        result["cpu_baseline_1thread"] = cpu_baseline(host, x_first, openmp=False)
    if world == 1 and not args.no_sub_records and args.config == WORKLOAD:
        # the other workloads of the suite, each with its own roofline, e2e
        # and oracle baseline (not timed into the headline)
        subs = []
        for name, k, w in SUB_RECORDS:
            sp = get_config(name)
            r, xf, ih = measure_layer(sp, k, w, rank, world, local)
            if sp.zipf_s is not None:
                r["routing_histogram"] = zipf_histogram(sp, ih)
            if not args.no_cpu_baseline:
                r["cpu_baseline"] = cpu_baseline(HostOracleLayer(sp, seed=0), xf, openmp=True)
            subs.append(r)
        for name, tokens in (("v3_stack20", 1), ("v3_stack20", 8), ("v3_stack20_ki", 1)):
            subs.append(measure_stack(get_config(name), tokens, 64, 5, rank, world, local,
                                      cpu=not args.no_cpu_baseline))
        result["sub_records"] = subs
    if world > 1:
        dist.barrier()
        dist.destroy_process_group()
    if result is not None:
        print(json.dumps(result))


def measure_stack(base, T, K, W, rank=0, world=1, local=0, cpu=True):
    """A stack of independent V3 layers (each with its own 192 mixed-format
    experts + shared expert, all resident in HBM); one step = one batch of
    fresh tokens through every layer, the layer calls captured once in a CUDA
    graph and replayed.  Weights per step (several GB) far exceed the L2, so no
    flush is needed between steps.  Returns the result dict (rank 0) or None."""
    import torch
    from workloads.synth import draw_tokens
    from dataclasses import replace

    import paper_2509_25689_gb300 as mq
    spec = replace(base, tokens=T)
    L = spec.n_layers
    P = spec.expert_param_count()
    ex = spec.extra
    if "k_orig" in ex:
        # per-layer activated experts k_i <= ceil(r k_orig) under the
        # workload's FLOPs budget (the library's activation plan)
        k_layers, _ = mq.mq_activation_plan(ex["k_orig"], ex["retain"], [P] * L, 2 * ex["budget_expert_acts"] * P)
        k_layers = [int(v) for v in k_layers]
    else:
        k_layers = [spec.top_k] * L
    kmax = max(k_layers)
    lspecs = [replace(spec, top_k=k_layers[l]) for l in range(L)]
    layers = [BenchLayer(lspecs[l], seed=1000 * rank + l) for l in range(L)]
    resident = sum(int(t.numel()) for lay in layers for trip in lay.tensors for t in trip)
    n_pool = max(1, min(W + K, (64 << 20) // (L * T * spec.hidden * 2)))
    x_host = np.stack([np.stack([draw_tokens(5000 + rank * 100003 + i * L + l, T, spec.hidden) for l in range(L)])
                       for i in range(n_pool)])                      # [pool, L, T, H] bf16 bits
    x_dev = torch.from_numpy(x_host.view(np.int16)).cuda()
    xbuf = torch.empty((L, T, spec.hidden), dtype=torch.int16, device="cuda")
    # layer l writes its [T, k_l] ids into its own region of one buffer
    idx_g = torch.full((L, T * kmax), -1, dtype=torch.int32, device="cuda")
    idx_views = [idx_g[l, :T * k_layers[l]].view(T, k_layers[l]) for l in range(L)]
    stream = torch.cuda.Stream()

    def eager():
        for l, lay in enumerate(layers):
            lay.forward(xbuf[l], idx_views[l])

    xbuf.copy_(x_dev[0])
    with torch.cuda.stream(stream):
        eager()                                  # first call outside capture (library set-up)
    torch.cuda.synchronize()
    graph = torch.cuda.CUDAGraph()
    with torch.cuda.graph(graph, stream=stream):
        eager()
    torch.cuda.synchronize()
    for i in range(W):
        xbuf.copy_(x_dev[i % n_pool])
        graph.replay()
    torch.cuda.synchronize()

    idx_steps = torch.empty((K, L, T * kmax), dtype=torch.int32, device="cuda")
    clocks = ClockSampler(local)
    clocks.start()
    evs = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(K)]
    torch.cuda.synchronize()
    t_wall0 = time.perf_counter()
    for i in range(K):
        evs[i][0].record()
        xbuf.copy_(x_dev[(W + i) % n_pool])
        graph.replay()
        idx_steps[i].copy_(idx_g)
        evs[i][1].record()
    torch.cuda.synchronize()
    t_wall = time.perf_counter() - t_wall0
    clk = clocks.stop()
    dev_ms = sum(a.elapsed_time(b) for a, b in evs)
    dev_ms_max = max_over_ranks(dev_ms, world, "cuda")

    # per-kernel durations: eager layer calls with an event pair per kernel
    layers[0].mq.mq_profile_enable(min(K, 8) * L * 8)
    for i in range(min(K, 8)):
        xbuf.copy_(x_dev[(W + i) % n_pool])
        eager()
    torch.cuda.synchronize()
    kstats = layers[0].mq.mq_profile_collect()

    # end to end: inputs from pinned host memory, every layer's output back
    x_pin = torch.from_numpy(x_host.view(np.int16)).pin_memory()
    outs = torch.stack([lay.out for lay in layers])           # refreshed per step below
    out_pin = torch.empty(tuple(outs.shape), dtype=torch.float32).pin_memory()
    e2e_evs = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(K)]
    torch.cuda.synchronize()
    for i in range(K):
        e2e_evs[i][0].record()
        xbuf.copy_(x_pin[(W + i) % n_pool], non_blocking=True)
        graph.replay()
        for l, lay in enumerate(layers):
            out_pin[l].copy_(lay.out, non_blocking=True)
        e2e_evs[i][1].record()
    torch.cuda.synchronize()
    e2e_ms = max_over_ranks(sum(a.elapsed_time(b) for a, b in e2e_evs), world, "cuda")

    idx_host = idx_steps.cpu().numpy()
    step_idx = lambda i, l: idx_host[i, l, :T * k_layers[l]].reshape(T, k_layers[l])
    touched = 0
    for i in range(K):
        for l, lay in enumerate(layers):
            sb = step_bytes(lspecs[l], lay.fmts, [step_idx(i, l)])[0]
            touched += sb["quantized"]
    peak, peak_src = _peaks()
    gbs = touched / (dev_ms / 1e3) / 1e9
    result = None
    if rank == 0:
        result = {
            "metric": METRIC, "value": round(job_throughput(world, T, K, dev_ms_max), 2), "unit": "tokens/s",
            "n_gpus": world, "steps": K, "warmup": W, "ms_per_step": round(dev_ms_max / K, 5),
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f16xf16->f32",
            "data": "synthetic (seeded random packed weights on device; fresh N(0,1) bf16 tokens per layer per step)",
            "config": {"workload": f"{spec.name}: {L} independent V3 layers (hidden {spec.hidden}, inter "
                                   f"{spec.inter}, {spec.n_experts} mixed-format experts + shared Q8_0 each), "
                                   f"T={T} per layer" + (f", k_i <= {kmax} per layer (activation plan for "
                                                         f"{ex['budget_expert_acts']} expert activations per token)"
                                                         if "k_orig" in ex else ""),
                       "resident_weight_bytes": resident,
                       "l2": "not flushed: each step reads several GB of weights (> 129 MB L2)",
                       "graph": f"the {L} layer calls captured once in a CUDA graph",
                       "parallelism": f"replicas x{world}"},
            "activated_experts_per_layer": k_layers,
            "flops_active_per_token": flops_active_per_token(k_layers, P, spec.has_shared),
            "activated_experts_per_layer": k_layers,
            "flops_active_per_token": flops_active_per_token(k_layers, P, spec.has_shared),
            "achieved_hbm_gbs": round(gbs, 1), "hbm_frac_of_measured": round(gbs / peak, 4),
            "hbm_frac_of_8tbs": round(gbs / 8000.0, 4), "quantized_bytes_per_step": int(touched / K),
            "kernels": [{"name": n, "launches": c, "total_ms": round(ms, 4)} for n, c, ms in kstats],
            "gpu_launches": int(L * sum(c for _, c, _ in kstats) / max(1, min(K, 8) * L)) * K,
            "wall_s_timed_region": round(t_wall, 4), "clocks": clk,
            "e2e": {"value": round(job_throughput(world, T, K, e2e_ms), 2), "unit": "tokens/s",
                    "h2d_bytes_per_step": int(L * T * spec.hidden * 2),
                    "d2h_bytes_per_step": int(L * T * spec.hidden * 4)},
        }
        dominant = max(kstats, key=lambda s: s[2]) if kstats else None
        if dominant:
            name, launches, tot_ms = dominant
            per_launch = sum(step_bytes(lspecs[l], lay.fmts, [step_idx(0, l)])[0].get(name, 0)
                             for l, lay in enumerate(layers)) / L
            avg_s = tot_ms / launches / 1e3
            result["roofline"] = {"bound": "hbm", "kernel": name, "achieved": round(per_launch / avg_s / 1e9, 1),
                                  "peak": peak, "unit": "GB/s", "frac": round(per_launch / avg_s / 1e9 / peak, 4),
                                  "traffic": None, "peak_source": peak_src,
                                  "algorithmic_bytes_per_launch": int(per_launch),
                                  "avg_launch_us": round(avg_s * 1e6, 2)}
        if world == 1 and cpu:
            host = HostOracleLayer(lspecs[0], seed=0)
            cb = cpu_baseline(host, x_host[0, 0], openmp=True)
            cb["value"] = cb["value"] / L      # a token goes through every layer
            cb["sample"] = (f"one layer of the stack (k = {k_layers[0]}), divided by its {L} layers: " +
                            cb["sample"])
            result["cpu_baseline"] = cb
    del layers, x_dev, xbuf, graph
    torch.cuda.empty_cache()
    return result


def run_stack(args):
    import torch
    from workloads import get_config
    local = int(os.environ.get("LOCAL_RANK", "0"))
    rank = int(os.environ.get("RANK", "0"))
    world = int(os.environ.get("WORLD_SIZE", "1"))
    torch.cuda.set_device(local)
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl")
    base = get_config(args.config)
    result = measure_stack(base, args.tokens if args.tokens else base.tokens, args.steps, args.warmup, rank, world,
                           local, cpu=not args.no_cpu_baseline)
    if result is not None:
        print(json.dumps(result))
    if world > 1:
        import torch.distributed as dist
        dist.barrier()
        dist.destroy_process_group()


def run_reference(args):
    """Reference arm: the oracle as it stands (its OpenMP build, identical
    results to the plain one) on the host cores, rank 0 only.  Every step is
    a fresh batch of the workload; the oracle is timed on a bounded sample of
    it and scaled to the whole batch (cpu_baseline), the run capped at about
    150 s of oracle time."""
    rank = int(os.environ.get("RANK", "0"))
    if rank != 0:
        return
    from workloads import get_config
    from workloads.synth import draw_tokens
    spec = get_config(args.config)
    T = args.tokens if (args.tokens and spec.n_layers > 1) else spec.tokens
    if T != spec.tokens:
        from dataclasses import replace
        spec = replace(spec, tokens=T)
    host = HostOracleLayer(spec, seed=0)
    budget_s, t_est, t_real, done_steps = 150.0, 0.0, 0.0, 0
    last = None
    for i in range(min(args.warmup, 1)):
        cpu_baseline(host, draw_tokens(1000 + i, T, spec.hidden), budget_s=4.0, openmp=True)
    for i in range(args.steps):
        w0 = time.perf_counter()
        last = cpu_baseline(host, draw_tokens(1000 + args.warmup + i, T, spec.hidden), budget_s=6.0, openmp=True)
        t_real += time.perf_counter() - w0
        t_est += T / last["value"]
        done_steps += 1
        if t_real > budget_s:
            break
    value = done_steps * T / t_est
    if spec.n_layers > 1:
        value /= spec.n_layers      # a token of the stack goes through every layer
    cb = dict(last)
    cb["value"] = round(value, 4)
    cb["sample"] = f"{done_steps} step(s); last: " + cb["sample"]
    line = {"metric": METRIC, "value": round(value, 4), "unit": "tokens/s", "n_gpus": 1, "steps": done_steps,
            "requested_steps": args.steps, "warmup": args.warmup,
            "ms_per_step": round(t_est / done_steps * 1e3 * (spec.n_layers if spec.n_layers > 1 else 1), 2),
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
            "data": "synthetic", "impl": "reference",
            "config": {"workload": f"{spec.name} (oracle: plain C, fp64 FFN, OpenMP build on {os.cpu_count()} "
                                   f"host cores" + (f"; one layer timed, value divided by the {spec.n_layers} "
                                                    f"layers)" if spec.n_layers > 1 else ")")},
            "cpu_baseline": cb,
            "e2e": {"value": round(value, 4), "unit": "tokens/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line))


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=2000)
    ap.add_argument("--warmup", type=int, default=20)
    ap.add_argument("--impl", default="native", choices=["native", "reference"])
    ap.add_argument("--config", default=WORKLOAD)
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-sub-records", action="store_true",
                    help="only the headline workload (no per-config sub-records)")
    ap.add_argument("--tokens", type=int, default=0, help="tokens per layer call for the layer-stack workload")
    args = ap.parse_args()
    if args.warmup < 3:
        args.warmup = 3
    from workloads import get_config
    if args.impl == "reference":
        run_reference(args)
    elif get_config(args.config).n_layers > 1:
        run_stack(args)
    else:
        run_native(args)


if __name__ == "__main__":
    main()
