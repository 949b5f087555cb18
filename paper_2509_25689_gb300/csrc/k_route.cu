// Router and permutation kernels.
//
// Router (arXiv 2509.25689 Sec. 3.2: sigmoid expert scores, topk_group
// groups over the pruned experts, num_experts_per_tok experts per token)
// in a canonical fp32 order so that expert ids are bit-exact with the CPU
// reference:
//   logit:   the row is cut in segments of 8 chunks x 128 elements; lane l
//            of the segment's warp runs one fma chain over chunk i, elements
//            128 i + 4 l + c (c = 0..3); an xor butterfly (16, 8, 4, 2, 1)
//            adds partners; segment results are added left to right.
//   sigmoid: Cody-Waite reduction a = n ln2 + r, degree-7 Taylor for e^r
//            (coefficients 1/i! rounded to fp32, Horner), exact 2^n scaling,
//            1/(1+e) with IEEE division; |a| clamped to 87.
//   select:  u = s + bias; group score = sum of the two largest u of a
//            group; keep topk_group groups, then top_k experts by u; ties go
//            to the lower index; weights s_j / sum(s) in slot order.
#include <cuda_runtime.h>
#include <stdint.h>

#include "mq_actprep.cuh"
#include "mq_internal.h"
#include "mq_select.cuh"

namespace mq {
namespace {

constexpr unsigned kFull = 0xffffffffu;

__device__ __forceinline__ float bf16_lo(uint32_t v) { return __uint_as_float(v << 16); }
__device__ __forceinline__ float bf16_hi(uint32_t v) { return __uint_as_float(v & 0xffff0000u); }

// Power-of-two exponent of a token's fp16 copy for the prefill GEMM: the
// token is stored as x * 2^-e with its largest magnitude in [1, 2), so any
// finite bf16 input fits the fp16 range (entries below 2^-24 of the largest
// become fp16 subnormals or zero, an error far below the fp32 accumulation's).
__device__ __forceinline__ int token_exp(float amax) { return amax > 0.0f ? ilogbf(amax) : 0; }

// ---------------------------------------------------------------------------
// logits for larger batches (no activation preparation): grid
// (ceil(E / kEB), ceil(T / kTokT)); a CTA keeps its 4 tokens' segments in
// registers as fp32 and runs through 16 experts, so the tokens are read and
// converted once per 16 experts instead of once per expert.  Same canonical
// order as router_logits_kernel (lane chains over the segment's chunks, xor
// butterfly, segments left to right), so z is bit-identical.
// ---------------------------------------------------------------------------
constexpr int kEB = 16;
constexpr int kTokT = 4;

__global__ void __launch_bounds__(256) router_logits_tile_kernel(const uint16_t* __restrict__ x,
                                                                  const float* __restrict__ W, int H, int T,
                                                                  int E, float* __restrict__ z,
                                                                  __half* __restrict__ x16, int32_t* __restrict__ xe) {
    __shared__ float part[8][kEB][kTokT];   // per segment (warp): each expert's sums of the CTA's tokens
    __shared__ float pmax[8][kTokT];        // per segment: largest |x| of each token (prefill copy)
    const int e0 = blockIdx.x * kEB, t0 = blockIdx.y * kTokT;
    const int seg = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int nchunk = H >> 7, nseg = (nchunk + 7) >> 3;
    const int c0 = seg * 8, nc = min(8, nchunk - c0);
    // the first expert's weights go out before the wait (an input no kernel of this library writes)
    float4 wv[8];
#pragma unroll
    for (int c = 0; c < 8; ++c)
        if (c < nc && e0 < E) wv[c] = __ldg(reinterpret_cast<const float4*>(W + (size_t)e0 * H + (c0 + c) * 128 + 4 * lane));
    pdl_wait();
    pdl_launch();
    float4 xf[kTokT][8];   // the tokens' segment elements 4 lane + 0..3 of each chunk, as fp32
#pragma unroll
    for (int j = 0; j < kTokT; ++j)
#pragma unroll
        for (int c = 0; c < 8; ++c) {
            uint2 v = make_uint2(0u, 0u);
            if (c < nc && t0 + j < T)
                v = __ldg(reinterpret_cast<const uint2*>(x + (size_t)(t0 + j) * H + (c0 + c) * 128 + 4 * lane));
            xf[j][c] = make_float4(bf16_lo(v.x), bf16_hi(v.x), bf16_lo(v.y), bf16_hi(v.y));
        }
    if (x16 != nullptr && blockIdx.x == 0) {
        // fp16 copy of the tokens for the prefill GEMM, each token scaled by
        // its power of two (the CTA holds its tokens' whole rows)
#pragma unroll
        for (int j = 0; j < kTokT; ++j) {
            float m = 0.0f;
#pragma unroll
            for (int c = 0; c < 8; ++c)
                m = fmaxf(m, fmaxf(fmaxf(fabsf(xf[j][c].x), fabsf(xf[j][c].y)), fmaxf(fabsf(xf[j][c].z), fabsf(xf[j][c].w))));
            m = warp_max_abs(m);
            if (lane == 0) pmax[seg][j] = m;
        }
        __syncthreads();
#pragma unroll
        for (int j = 0; j < kTokT; ++j) {
            if (t0 + j >= T) break;
            float m = pmax[0][j];
            for (int s2 = 1; s2 < nseg; ++s2) m = fmaxf(m, pmax[s2][j]);
            const int ex = token_exp(m);
            if (threadIdx.x == 0) xe[t0 + j] = ex;
#pragma unroll
            for (int c = 0; c < 8; ++c) {
                if (c >= nc) break;
                const __half2 h0 = __floats2half2_rn(ldexpf(xf[j][c].x, -ex), ldexpf(xf[j][c].y, -ex));
                const __half2 h1 = __floats2half2_rn(ldexpf(xf[j][c].z, -ex), ldexpf(xf[j][c].w, -ex));
                uint2 hv;
                hv.x = *reinterpret_cast<const uint32_t*>(&h0);
                hv.y = *reinterpret_cast<const uint32_t*>(&h1);
                *reinterpret_cast<uint2*>(x16 + (size_t)(t0 + j) * H + (c0 + c) * 128 + 4 * lane) = hv;
            }
        }
    }
    // expert el's weights in wv, expert el + 1's loading into wn while el is
    // reduced; the per-warp sums of all 16 experts wait in shared memory and
    // the segments are added once at the end
    for (int el = 0; el < kEB; ++el) {
        const int e = e0 + el;
        if (e >= E) break;
        float4 wn[8] = {};
        if (e + 1 < E && el + 1 < kEB) {
#pragma unroll
            for (int c = 0; c < 8; ++c)
                if (c < nc) wn[c] = __ldg(reinterpret_cast<const float4*>(W + (size_t)(e + 1) * H + (c0 + c) * 128 + 4 * lane));
        }
        float acc[kTokT];
#pragma unroll
        for (int j = 0; j < kTokT; ++j) {
            acc[j] = 0.0f;
#pragma unroll
            for (int c = 0; c < 8; ++c) {
                if (c < nc) {
                    acc[j] = __fmaf_rn(xf[j][c].x, wv[c].x, acc[j]);
                    acc[j] = __fmaf_rn(xf[j][c].y, wv[c].y, acc[j]);
                    acc[j] = __fmaf_rn(xf[j][c].z, wv[c].z, acc[j]);
                    acc[j] = __fmaf_rn(xf[j][c].w, wv[c].w, acc[j]);
                }
            }
        }
#pragma unroll
        for (int j = 0; j < kTokT; ++j) {
#pragma unroll
            for (int off = 16; off >= 1; off >>= 1) acc[j] = __fadd_rn(acc[j], __shfl_xor_sync(kFull, acc[j], off));
        }
        if (lane == 0) {
#pragma unroll
            for (int j = 0; j < kTokT; ++j) part[seg][el][j] = acc[j];
        }
#pragma unroll
        for (int c = 0; c < 8; ++c) wv[c] = wn[c];
    }
    __syncthreads();
    // segments left to right, per (expert, token) of the CTA
    for (int o = threadIdx.x; o < kEB * kTokT; o += blockDim.x) {
        const int el = o / kTokT, j = o % kTokT, e = e0 + el, t = t0 + j;
        if (e < E && t < T) {
            float r = part[0][el][j];
            for (int s2 = 1; s2 < nseg; ++s2) r = __fadd_rn(r, part[s2][el][j]);
            z[(size_t)t * E + e] = r;
        }
    }
}

// Per-call words that must start at zero (work counters, the h and routing
// flags, the error word), cleared by the first kernel of a forward call.  It
// lets its successor launch at once (that kernel waits for this one before
// touching the words) and itself waits for the previous kernel on the
// stream, so the previous call no longer uses them.
__global__ void zero_kernel(uint32_t* __restrict__ words, int n) {
    pdl_launch();
    pdl_wait();
    for (int i = threadIdx.x; i < n; i += blockDim.x) words[i] = 0u;
}

constexpr int kTopkWarps = 4;

__global__ void __launch_bounds__(kTopkWarps * 32) topk_kernel(const float* __restrict__ z,
                                                               const float* __restrict__ bias, Dims d,
                                                               int32_t* __restrict__ idx,
                                                               float* __restrict__ wts) {
    __shared__ float u_sh[kTopkWarps][kMaxExperts];
    __shared__ float g_sh[kTopkWarps][kMaxGroups];
    pdl_wait();
    pdl_launch();
    const int w = threadIdx.x >> 5;
    const int t = blockIdx.x * kTopkWarps + w;
    if (t >= d.T) return;
    sel::route_token(z, bias, d.E, d.G, d.Gk, d.K, d.routed_scale, t, u_sh[w], g_sh[w], idx, wts);
}

// ---------------------------------------------------------------------------
// permutation: one CTA; stable counting sort of entries a = t*K + j by expert
// ---------------------------------------------------------------------------
constexpr int kPermThreads = 512;
constexpr int kPermWarps = kPermThreads / 32;
// barrier 2 over the kPermThreads routing threads (the CTA may have more)
__device__ __forceinline__ void perm_sync() { asm volatile("bar.sync 2, %0;" ::"n"(kPermThreads) : "memory"); }

// Shared memory of the routing + permutation step (one CTA).
struct PermSmem {
    int32_t cnt[kPermWarps][kMaxExperts];   // per-warp segment counts, then cursors
    int32_t s_off[kMaxExperts + 1];
    int32_t s_act[kMaxExperts + 1];
    float g_sh[kPermWarps][kMaxGroups];
    float s_bias[kMaxExperts];
};

// Routing and permutation by the first kPermThreads threads of one CTA (the
// caller has staged the selection bias in S.s_bias and synchronised).  With
// `z` given, the CTA first routes every token (one warp per token,
// decode-sized batches) and then permutes.  Offsets and the active list are
// kept in shared memory as well, so nothing written here is read back from
// global memory.  offsets, inv and active may be NULL (not written).  Threads
// leave by returning; block-wide steps use a named barrier over the
// kPermThreads threads, so the CTA may hold more.  route_warp: the warp that
// routes a single token (the others return at once on that path).
__device__ void route_permute_cta(PermSmem& S, int32_t* __restrict__ idx, const Dims& d,
                                  int32_t* __restrict__ offsets, int32_t* __restrict__ perm,
                                  int32_t* __restrict__ inv, int32_t* __restrict__ active,
                                  Plan* __restrict__ plan, const float* __restrict__ z,
                                  float* __restrict__ wts, int route_warp = 0) {
    const int n = d.T * d.K, E = d.E;
    auto& cnt = S.cnt;
    auto& s_off = S.s_off;
    auto& s_act = S.s_act;
    auto& g_sh = S.g_sh;
    const float* s_bias = S.s_bias;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    if (warp >= kPermWarps) return;
    if (z != nullptr && d.T == 1 && d.K <= 32 && E <= 256) {
        // One token: the selection holds K distinct experts, one entry each, so
        // the counting sort reduces to ranking them.  One warp does all of it
        // in registers (no block barriers, nothing read back from global memory).
        if (warp != route_warp) return;
        const int K = d.K;
        int sel = 0;
        // scratch: rows 0 and 1 of the counting table (free on this path)
        sel::route_token_compact(z, s_bias, d.E, d.G, d.Gk, K, d.routed_scale, 0, reinterpret_cast<float*>(cnt[0]),
                                 g_sh[route_warp], idx, wts, &sel);
        // the selection as a 256-bit set; an expert's rank (and offsets[e]) is
        // the number of selected ids below it
        uint32_t mask[8];
#pragma unroll
        for (int w = 0; w < 8; ++w)
            mask[w] = __reduce_or_sync(kFull, (lane < K && (sel >> 5) == w) ? 1u << (sel & 31) : 0u);
        auto below = [&](int e) {   // selected ids < e (e <= 256)
            int c = 0;
#pragma unroll
            for (int w = 0; w < 8; ++w)
                c += __popc(32 * w + 32 <= e ? mask[w] : (32 * w < e ? mask[w] & ((1u << (e & 31)) - 1u) : 0u));
            return c;
        };
        const int rank = below(sel);
        if (lane < K) {
            perm[rank] = lane;   // entry a = t * K + j = j
            if (inv) inv[lane] = rank;
            if (active) active[1 + rank] = sel;
        }
        if (lane == 0 && active) active[0] = K;
        // offsets[e] = selected experts with a lower id; offsets[E] = K
        if (offsets) {
#pragma unroll
            for (int q = 0; q < 8; ++q) {
                const int e = lane * 8 + q;
                if (e < E) offsets[e] = below(e);
            }
            if (lane == 0) offsets[E] = K;
        }
        if (plan == nullptr) return;
        // work plan: slot p (shared expert first) holds one token
        const int n_slots = K + d.has_shared;
        for (int p = lane; p <= kMaxExperts + 1; p += 32) {
            const int pc = min(p, n_slots);
            plan->pre_gu[p] = pc * (d.I / 32);
            plan->pre_dn[p] = pc * (d.H / 64);
        }
        // slot of the expert of rank r: has_shared + r
        if (lane < K) {
            const int p = d.has_shared + rank;
            plan->slot_e[p] = sel;
            plan->slot_first[p] = rank;
            plan->slot_ntot[p] = 1;
        }
        if (lane == 0) {
            if (d.has_shared) { plan->slot_e[0] = d.E; plan->slot_first[0] = 0; plan->slot_ntot[0] = 1; }
            plan->n_slots = n_slots;
            plan->dn_target = n_slots;
            plan->ntg_max = 1;
        }
        return;
    }
    if (z != nullptr) {
        for (int t = warp; t < d.T; t += kPermWarps)
            sel::route_token(z, s_bias, d.E, d.G, d.Gk, d.K, d.routed_scale, t, reinterpret_cast<float*>(cnt[warp]),
                        g_sh[warp], idx, wts);
        perm_sync();
    }
    for (int i = threadIdx.x; i < kPermWarps * kMaxExperts; i += kPermThreads) (&cnt[0][0])[i] = 0;
    perm_sync();
    const int seg = (n + kPermWarps - 1) / kPermWarps;
    const int a0 = warp * seg, a1 = min(n, a0 + seg);
    for (int a = a0 + lane; a < a1; a += 32) atomicAdd(&cnt[warp][idx[a]], 1);
    perm_sync();
    // per-expert totals and per-warp starting cursors (warp order = entry order)
    if (threadIdx.x < E) {
        const int e = threadIdx.x;
        int run = 0;
#pragma unroll
        for (int wv = 0; wv < kPermWarps; ++wv) { const int c = cnt[wv][e]; cnt[wv][e] = run; run += c; }
        s_off[e] = run;
    }
    perm_sync();
    if (warp == 0) {
        // exclusive scan of totals over experts (E <= 256: 8 per lane)
        int local[8], sum = 0;
#pragma unroll
        for (int q = 0; q < 8; ++q) {
            const int e = lane * 8 + q;
            local[q] = e < E ? s_off[e] : 0;
            sum += local[q];
        }
        int incl = sum;
#pragma unroll
        for (int off = 1; off < 32; off <<= 1) {
            const int v = __shfl_up_sync(kFull, incl, off);
            if (lane >= off) incl += v;
        }
        int run = incl - sum;
        __syncwarp();
#pragma unroll
        for (int q = 0; q < 8; ++q) {
            const int e = lane * 8 + q;
            if (e < E) { if (offsets) offsets[e] = run; s_off[e] = run; }
            run += local[q];
        }
        if (lane == 31) { if (offsets) offsets[E] = run; s_off[E] = run; }
    }
    perm_sync();
    for (int i = threadIdx.x; i < kPermWarps * E; i += kPermThreads) {
        const int wv = i / E, e = i - wv * E;
        cnt[wv][e] += s_off[e];
    }
    perm_sync();
    // stable scatter: each warp walks its segment in order, 32 entries a step
    for (int base = a0; base < a1; base += 32) {
        const int a = base + lane;
        const bool ok = a < a1;
        const int e = ok ? idx[a] : -1 - lane;
        const unsigned peers = __match_any_sync(kFull, e);
        const int rank = __popc(peers & ((1u << lane) - 1u));
        if (ok) {
            const int pos = cnt[warp][e] + rank;
            perm[pos] = a;
            if (inv) inv[a] = pos;
        }
        __syncwarp();
        if (ok && rank == 0) cnt[warp][e] += __popc(peers);
        __syncwarp();
    }
    // active expert list (ascending ids), active[0] = count
    if (warp == 0) {
        int flags = 0, c = 0;
#pragma unroll
        for (int q = 0; q < 8; ++q) {
            const int e = lane * 8 + q;
            const int f = (e < E && s_off[e + 1] > s_off[e]) ? 1 : 0;
            flags |= f << q;
            c += f;
        }
        int incl = c;
#pragma unroll
        for (int off = 1; off < 32; off <<= 1) {
            const int v = __shfl_up_sync(kFull, incl, off);
            if (lane >= off) incl += v;
        }
        int pos = incl - c;
#pragma unroll
        for (int q = 0; q < 8; ++q)
            if (flags & (1 << q)) { if (active) active[1 + pos] = lane * 8 + q; s_act[1 + pos] = lane * 8 + q; ++pos; }
        if (lane == 31) { if (active) active[0] = incl; s_act[0] = incl; }
    }
    if (plan == nullptr) return;
    perm_sync();
    // decode work plan: items per expert slot (shared expert first)
    if (warp == 0) {
        const int n_slots = s_act[0] + d.has_shared;
        int cg[9], cd[9], sg = 0, sd = 0, tgs = 0, tgmax = 0;
#pragma unroll
        for (int q = 0; q < 9; ++q) {
            const int p = lane * 9 + q;
            int ntok = 0, e = d.E, first = 0;
            if (p < n_slots) {
                if (p < d.has_shared) ntok = d.T;
                else { e = s_act[1 + p - d.has_shared]; first = s_off[e]; ntok = s_off[e + 1] - first; }
                plan->slot_e[p] = e;
                plan->slot_first[p] = first;
                plan->slot_ntot[p] = ntok;
            }
            const int ntg = (ntok + kDecodeTok - 1) / kDecodeTok;
            cg[q] = (d.I / 32) * ntg;     // gate/up items: 32 rows x both tensors x full K
            cd[q] = (d.H / 64) * ntg;     // down items: 64 rows (two 32-row blocks) x full K
            sg += cg[q]; sd += cd[q]; tgs += ntg; tgmax = max(tgmax, ntg);
        }
        int ig = sg, id = sd;
#pragma unroll
        for (int off = 1; off < 32; off <<= 1) {
            const int vg = __shfl_up_sync(kFull, ig, off), vd = __shfl_up_sync(kFull, id, off);
            if (lane >= off) { ig += vg; id += vd; }
        }
        int rg = ig - sg, rd = id - sd;
#pragma unroll
        for (int q = 0; q < 9; ++q) {
            const int p = lane * 9 + q;
            if (p <= kMaxExperts + 1) { plan->pre_gu[p] = rg; plan->pre_dn[p] = rd; }
            rg += cg[q]; rd += cd[q];
        }
#pragma unroll
        for (int off = 16; off >= 1; off >>= 1) {
            tgs += __shfl_xor_sync(kFull, tgs, off);
            tgmax = max(tgmax, __shfl_xor_sync(kFull, tgmax, off));
        }
        if (lane == 0) {
            plan->n_slots = n_slots;
            plan->dn_target = tgs;
            plan->ntg_max = tgmax;
        }
    }
}

// Standalone routing + permutation kernel (one CTA of kPermThreads).
__global__ void __launch_bounds__(kPermThreads) permute_kernel(int32_t* __restrict__ idx, Dims d,
                                                               int32_t* __restrict__ offsets,
                                                               int32_t* __restrict__ perm,
                                                               int32_t* __restrict__ inv,
                                                               int32_t* __restrict__ active,
                                                               Plan* __restrict__ plan,
                                                               const float* __restrict__ z,
                                                               const float* __restrict__ bias,
                                                               float* __restrict__ wts) {
    __shared__ PermSmem S;
    // the selection bias is an input no kernel of this library writes: staged
    // before the wait for the logits kernel
    if (z != nullptr)
        for (int i = threadIdx.x; i < d.E; i += kPermThreads) S.s_bias[i] = bias ? bias[i] : 0.0f;
    __syncthreads();
    pdl_wait();
    pdl_launch();
    route_permute_cta(S, idx, d, offsets, perm, inv, active, plan, z, wts);
}

// ---------------------------------------------------------------------------
// logits: grid (ceil(E / epc), ceil(T / kTok)); a CTA holds epc experts, one
// warp per (expert, 1024-element segment), so that at decode most SMs hold
// no logits CTA and take the expert-FFN grid (which needs a whole SM's shared
// memory) as soon as it launches.  Every expert's sum is formed in the same
// canonical order whatever epc is.
// ---------------------------------------------------------------------------
constexpr int kTok = 8;
#ifndef MQ_LOGITS_EPC
#define MQ_LOGITS_EPC 1
#endif
constexpr int kLogitsEpc = MQ_LOGITS_EPC;   // experts per logits CTA (fewer if the warps would exceed 32)

__host__ __device__ __forceinline__ int logits_nseg(int H) { return (H / 128 + 7) / 8; }
__host__ __device__ __forceinline__ int logits_epc(int H) {
    const int nseg = logits_nseg(H);
    const int e = 32 / (nseg > 0 ? nseg : 1);
    return e < 1 ? 1 : (e > kLogitsEpc ? kLogitsEpc : e);
}

__global__ void __launch_bounds__(1024) router_logits_kernel(const uint16_t* __restrict__ x,
                                                             const float* __restrict__ W, int H, int T,
                                                             int E, float* __restrict__ z,
                                                             __half* __restrict__ xq, float* __restrict__ xs,
                                                             __half* __restrict__ x16, int32_t* __restrict__ xe,
                                                             int x_fams, int epc, const FusedRoute fr) {
    __shared__ float part[32][kTok];
    __shared__ float pmax[32][kTok];   // per warp: largest |x| of each token (prefill copy only)
    __shared__ int s_last;
    const int t0 = blockIdx.y * kTok;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int nchunk = H >> 7, nseg = (nchunk + 7) >> 3;
    // warp -> (local expert le, segment seg); warps past epc experts (the
    // routing CTA's extra warps) and experts past E take no segment
    const int le = warp / nseg, seg = warp - le * nseg;
    const int e = blockIdx.x * epc + le;
    const bool work = le < epc && e < E;
    const int c0 = seg * 8, nc = work ? min(8, nchunk - c0) : 0;
    const float* wrow = W + (size_t)(work ? e : 0) * H;
    // The router weights are an input no kernel of this library writes, so
    // their loads go out before the wait for the previous kernel (which may
    // be the previous layer's combine, writing this call's x).
    float4 wv[8];
#pragma unroll
    for (int c = 0; c < 8; ++c)
        if (c < nc) wv[c] = __ldg(reinterpret_cast<const float4*>(wrow + (c0 + c) * 128 + 4 * lane));
    // fused routing: every CTA stages the selection bias (an input as well)
    // now, so the CTA that ends up routing has it without another round trip
    extern __shared__ __align__(16) uint8_t dyn_smem[];
    PermSmem& S = *reinterpret_cast<PermSmem*>(dyn_smem);
    if (fr.on) {
        for (int i = threadIdx.x; i < E; i += blockDim.x) S.s_bias[i] = fr.bias ? __ldg(fr.bias + i) : 0.0f;
        __syncthreads();
    }
    pdl_wait();
    pdl_launch();
    float acc[kTok], amx[kTok];
#pragma unroll
    for (int j = 0; j < kTok; ++j) acc[j] = amx[j] = 0.0f;
#pragma unroll
    for (int j = 0; j < kTok; ++j) {
        const int t = t0 + j;
        if (t >= T) break;
        const uint16_t* xr = x + (size_t)t * H;
#pragma unroll
        for (int c = 0; c < 8; ++c) {
            if (c < nc) {
                const uint2 xv = __ldg(reinterpret_cast<const uint2*>(xr + (c0 + c) * 128 + 4 * lane));
                acc[j] = __fmaf_rn(bf16_lo(xv.x), wv[c].x, acc[j]);
                acc[j] = __fmaf_rn(bf16_hi(xv.x), wv[c].y, acc[j]);
                acc[j] = __fmaf_rn(bf16_lo(xv.y), wv[c].z, acc[j]);
                acc[j] = __fmaf_rn(bf16_hi(xv.y), wv[c].w, acc[j]);
                if (x16 != nullptr)
                    amx[j] = fmaxf(amx[j], fmaxf(fmaxf(fabsf(bf16_lo(xv.x)), fabsf(bf16_hi(xv.x))),
                                                 fmaxf(fabsf(bf16_lo(xv.y)), fabsf(bf16_hi(xv.y)))));
            }
        }
    }
#pragma unroll
    for (int j = 0; j < kTok; ++j) {
#pragma unroll
        for (int off = 16; off >= 1; off >>= 1) acc[j] = __fadd_rn(acc[j], __shfl_xor_sync(kFull, acc[j], off));
        if (x16 != nullptr) amx[j] = warp_max_abs(amx[j]);
    }
    if (lane == 0) {
#pragma unroll
        for (int j = 0; j < kTok; ++j) { part[warp][j] = acc[j]; pmax[warp][j] = amx[j]; }
    }
    __syncthreads();
    // z: per (local expert, token), the expert's segments left to right
    if (threadIdx.x < epc * kTok) {
        const int l2 = threadIdx.x / kTok, j = threadIdx.x - l2 * kTok;
        const int e2 = blockIdx.x * epc + l2, t = t0 + j;
        if (e2 < E && t < T) {
            float r = part[l2 * nseg][j];
            for (int s = 1; s < nseg; ++s) r = __fadd_rn(r, part[l2 * nseg + s][j]);
            z[(size_t)t * E + e2] = r;
        }
    }
    // fp16 copy of the tokens for the prefill GEMM (each token scaled by its
    // power of two), spread over the CTAs
    if (x16 != nullptr) {
        for (int j = 0; j < kTok; ++j) {
            const int t = t0 + j;
            if (t >= T) break;
            // the CTA's first expert's warps saw the whole token
            float m = pmax[0][j];
            for (int s = 1; s < nseg; ++s) m = fmaxf(m, pmax[s][j]);
            const int ex = token_exp(m);
            if (blockIdx.x == 0 && threadIdx.x == 0) xe[t] = ex;
            for (int k = blockIdx.x * blockDim.x + threadIdx.x; k < H; k += gridDim.x * blockDim.x)
                x16[(size_t)t * H + k] = __float2half_rn(ldexpf(bf16_lo(x[(size_t)t * H + k]), -ex));
        }
    }
    // The CTAs also prepare the tokens' activations for the expert-FFN
    // kernels, spread over all of them: warp `seg` of the CTA of expert e
    // takes the 32-element blocks 32*seg + e, 32*seg + e + E, ... of its
    // segment (blocks past the hidden size, up to the 256 padding, are zero).
    if (xq != nullptr && work) {
        const int nsb = (H + 255) / 256;
        const size_t qstride = (size_t)kFamSlots * nsb * 256, sstride = (size_t)nsb * kStatFloats;
        for (int j = 0; j < kTok; ++j) {
            const int t = t0 + j;
            if (t >= T) break;
            for (int jb = 32 * seg + e; jb < 32 * seg + 32 && jb < 8 * nsb; jb += E) {
                const int k = 32 * jb + lane;
                const float v = k < H ? bf16_lo(x[(size_t)t * H + k]) : 0.0f;
                prep_block32(v, jb, x_fams, xq + (size_t)t * qstride,
                             xs + (size_t)t * sstride, nsb);
            }
        }
    }
    if (!fr.on) return;
    // Routing fused in: every CTA publishes its logits and prepared tokens
    // with one acquire-release count (the block barrier orders every
    // thread's stores before thread 0's count); the CTA that counts last has
    // acquired every other CTA's stores with it, routes every token and
    // permutes, then publishes the result with a release store.  The
    // expert-FFN kernel, launched as this grid's dependent, waits on the
    // count (prepared tokens) and on the release flag (routing result).
    __syncthreads();
    if (threadIdx.x == 0) {
        uint32_t old;
        asm volatile("atom.acq_rel.gpu.global.add.u32 %0, [%1], 1;" : "=r"(old) : "l"(fr.logits_done) : "memory");
        s_last = old == fr.n_ctas - 1u;
    }
    __syncthreads();
    if (!s_last) return;
    route_permute_cta(S, fr.idx, fr.d, fr.offsets, fr.perm, fr.inv, fr.active, fr.plan, z, fr.wts);
    __syncthreads();
    if (threadIdx.x == 0) asm volatile("st.release.gpu.global.u32 [%0], %1;" ::"l"(fr.route_ready), "r"(1u) : "memory");
}


void route_setup() {
    prefer_max_shared(router_logits_kernel);
    prefer_max_shared(router_logits_tile_kernel);
    prefer_max_shared(topk_kernel);
    prefer_max_shared(permute_kernel);
}

}  // namespace

cudaError_t launch_zero(uint32_t* words, int n, cudaStream_t s) {
    prof_begin("zero", s);
    const cudaError_t e = launch_pdl(zero_kernel, dim3(1), dim3(256), 0, s, words, n);
    prof_end(s);
    return e;
}

uint32_t router_logits_ctas(const Dims& d) {
    const int epc = logits_epc(d.H);
    return (uint32_t)(((d.E + epc - 1) / epc) * ((d.T + kTok - 1) / kTok));
}

cudaError_t launch_router_logits(const Dims& d, const uint16_t* x, const float* W, float* z, __half* xq, float* xs,
                                 __half* x16, int32_t* xe, const FusedRoute* fused, cudaStream_t s) {
    if (d.T == 0) return cudaSuccess;
    const int nseg = (d.H / 128 + 7) / 8;
    if (device_setup(kSetupRoute, route_setup) <= 0) return cudaErrorInvalidDevice;
    prof_begin("router_logits", s);
    cudaError_t e;
    if (fused == nullptr && xq == nullptr && d.T >= 16 && nseg <= 8) {
        // larger batches without activation preparation: tokens reused across 16 experts
        dim3 grid((d.E + kEB - 1) / kEB, (d.T + kTokT - 1) / kTokT);
        e = launch_pdl(router_logits_tile_kernel, grid, dim3(nseg * 32), 0, s, x, W, d.H, d.T, d.E, z, x16, xe);
    } else {
        const int epc = logits_epc(d.H);
        dim3 grid((d.E + epc - 1) / epc, (d.T + kTok - 1) / kTok);
        FusedRoute fr{};
        int warps = epc * nseg;
        size_t smem = 0;
        if (fused != nullptr) {
            fr = *fused;
            fr.on = 1;
            fr.n_ctas = grid.x * grid.y;
            if (warps < kPermWarps) warps = kPermWarps;   // the last CTA routes with kPermWarps warps
            smem = sizeof(PermSmem);
        }
        e = launch_pdl(router_logits_kernel, grid, dim3(warps * 32), smem, s, x, W, d.H, d.T, d.E, z, xq, xs, x16,
                       xe, d.x_fams, epc, fr);
    }
    prof_end(s);
    return e;
}

cudaError_t launch_topk(const Dims& d, const float* z, const float* bias, int32_t* idx, float* wts,
                        cudaStream_t s) {
    if (d.T == 0) return cudaSuccess;
    if (device_setup(kSetupRoute, route_setup) <= 0) return cudaErrorInvalidDevice;
    prof_begin("router_topk", s);
    const cudaError_t e = launch_pdl(topk_kernel, dim3((d.T + kTopkWarps - 1) / kTopkWarps), dim3(kTopkWarps * 32),
                                     0, s, z, bias, d, idx, wts);
    prof_end(s);
    return e;
}

cudaError_t launch_permute(const Dims& d, const int32_t* idx, int32_t* offsets, int32_t* perm, int32_t* inv,
                           int32_t* active, Plan* plan, cudaStream_t s) {
    if (device_setup(kSetupRoute, route_setup) <= 0) return cudaErrorInvalidDevice;
    prof_begin("permute", s);
    const cudaError_t e = launch_pdl(permute_kernel, dim3(1), dim3(kPermThreads), 0, s, const_cast<int32_t*>(idx), d,
                                     offsets, perm, inv, active, plan, (const float*)nullptr, (const float*)nullptr,
                                     (float*)nullptr);
    prof_end(s);
    return e;
}

cudaError_t launch_route_permute(const Dims& d, const float* z, const float* bias, int32_t* idx, float* wts,
                                 int32_t* offsets, int32_t* perm, int32_t* inv, int32_t* active, Plan* plan,
                                 cudaStream_t s) {
    if (device_setup(kSetupRoute, route_setup) <= 0) return cudaErrorInvalidDevice;
    prof_begin("route_permute", s);
    const cudaError_t e = launch_pdl(permute_kernel, dim3(1), dim3(kPermThreads), 0, s, idx, d, offsets, perm, inv,
                                     active, plan, z, bias, wts);
    prof_end(s);
    return e;
}

}  // namespace mq
