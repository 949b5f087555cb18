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

namespace mq {
namespace {

constexpr unsigned kFull = 0xffffffffu;

__device__ __forceinline__ float bf16_lo(uint32_t v) { return __uint_as_float(v << 16); }
__device__ __forceinline__ float bf16_hi(uint32_t v) { return __uint_as_float(v & 0xffff0000u); }

// ---------------------------------------------------------------------------
// logits: grid (E, ceil(T / kTok)), one warp per 1024-element segment
// ---------------------------------------------------------------------------
constexpr int kTok = 8;

__global__ void __launch_bounds__(1024) router_logits_kernel(const uint16_t* __restrict__ x,
                                                             const float* __restrict__ W, int H, int T,
                                                             int E, float* __restrict__ z,
                                                             __half* __restrict__ xq, float* __restrict__ xs,
                                                             __half* __restrict__ x16,
                                                             uint32_t* __restrict__ zero_words, int n_zero) {
    __shared__ float part[32][kTok];
    const int e = blockIdx.x, t0 = blockIdx.y * kTok;
    const int seg = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int nchunk = H >> 7, nseg = (nchunk + 7) >> 3;
    const int c0 = seg * 8, nc = min(8, nchunk - c0);
    const float* wrow = W + (size_t)e * H;
    // The router weights are an input no kernel of this library writes, so
    // their loads go out before the wait for the previous kernel (which may
    // be the previous layer's combine, writing this call's x).
    float4 wv[8];
#pragma unroll
    for (int c = 0; c < 8; ++c)
        if (c < nc) wv[c] = __ldg(reinterpret_cast<const float4*>(wrow + (c0 + c) * 128 + 4 * lane));
    pdl_wait();
    pdl_launch();
    // per-call words that must start at zero (work counters, error word)
    if (blockIdx.x == 0 && blockIdx.y == 0)
        for (int i = threadIdx.x; i < n_zero; i += blockDim.x) zero_words[i] = 0u;
    float acc[kTok];
#pragma unroll
    for (int j = 0; j < kTok; ++j) acc[j] = 0.0f;
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
            }
        }
    }
#pragma unroll
    for (int j = 0; j < kTok; ++j) {
#pragma unroll
        for (int off = 16; off >= 1; off >>= 1) acc[j] = __fadd_rn(acc[j], __shfl_xor_sync(kFull, acc[j], off));
    }
    if (lane == 0) {
#pragma unroll
        for (int j = 0; j < kTok; ++j) part[seg][j] = acc[j];
    }
    __syncthreads();
    if (threadIdx.x < kTok) {
        const int t = t0 + threadIdx.x;
        if (t < T) {
            float r = part[0][threadIdx.x];
            for (int s = 1; s < nseg; ++s) r = __fadd_rn(r, part[s][threadIdx.x]);
            z[(size_t)t * E + e] = r;
        }
    }
    // fp16 copy of the tokens for the prefill GEMM, spread over the CTAs
    if (x16 != nullptr) {
        for (int j = 0; j < kTok; ++j) {
            const int t = t0 + j;
            if (t >= T) break;
            for (int k = e * blockDim.x + threadIdx.x; k < H; k += E * blockDim.x)
                x16[(size_t)t * H + k] = __float2half_rn(bf16_lo(x[(size_t)t * H + k]));
        }
    }
    // The CTAs also prepare the tokens' activations for the expert-FFN
    // kernels, spread over all of them: warp `seg` of the CTA of expert e
    // takes the 32-element blocks 32*seg + e, 32*seg + e + E, ... of its
    // segment (blocks past the hidden size, up to the 256 padding, are zero).
    if (xq != nullptr) {
        const int nsb = (H + 255) / 256;
        const size_t qstride = (size_t)4 * nsb * 256, sstride = (size_t)nsb * kStatFloats;
        for (int j = 0; j < kTok; ++j) {
            const int t = t0 + j;
            if (t >= T) break;
            for (int jb = 32 * seg + e; jb < 32 * seg + 32 && jb < 8 * nsb; jb += E) {
                const int k = 32 * jb + lane;
                const float v = k < H ? bf16_lo(x[(size_t)t * H + k]) : 0.0f;
                prep_block32(v, jb, 0xF, xq + (size_t)t * qstride, xs + (size_t)t * sstride, nsb);
            }
        }
    }
}

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
                                                                  __half* __restrict__ x16,
                                                                  uint32_t* __restrict__ zero_words, int n_zero) {
    __shared__ float part[32][kTokT];
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
    if (blockIdx.x == 0 && blockIdx.y == 0)
        for (int i = threadIdx.x; i < n_zero; i += blockDim.x) zero_words[i] = 0u;
    float4 xf[kTokT][8];   // the tokens' segment elements 4 lane + 0..3 of each chunk, as fp32
#pragma unroll
    for (int j = 0; j < kTokT; ++j)
#pragma unroll
        for (int c = 0; c < 8; ++c) {
            uint2 v = make_uint2(0u, 0u);
            if (c < nc && t0 + j < T)
                v = __ldg(reinterpret_cast<const uint2*>(x + (size_t)(t0 + j) * H + (c0 + c) * 128 + 4 * lane));
            xf[j][c] = make_float4(bf16_lo(v.x), bf16_hi(v.x), bf16_lo(v.y), bf16_hi(v.y));
            if (x16 != nullptr && blockIdx.x == 0 && c < nc && t0 + j < T) {
                // fp16 copy of the tokens for the prefill GEMM
                const __half2 h0 = __floats2half2_rn(xf[j][c].x, xf[j][c].y);
                const __half2 h1 = __floats2half2_rn(xf[j][c].z, xf[j][c].w);
                uint2 hv;
                hv.x = *reinterpret_cast<const uint32_t*>(&h0);
                hv.y = *reinterpret_cast<const uint32_t*>(&h1);
                *reinterpret_cast<uint2*>(x16 + (size_t)(t0 + j) * H + (c0 + c) * 128 + 4 * lane) = hv;
            }
        }
    for (int el = 0; el < kEB; ++el) {
        const int e = e0 + el;
        if (e >= E) break;
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
        // the next expert's weights, loaded while this one's sums are reduced
        if (e + 1 < E && el + 1 < kEB) {
#pragma unroll
            for (int c = 0; c < 8; ++c)
                if (c < nc) wv[c] = __ldg(reinterpret_cast<const float4*>(W + (size_t)(e + 1) * H + (c0 + c) * 128 + 4 * lane));
        }
#pragma unroll
        for (int j = 0; j < kTokT; ++j) {
#pragma unroll
            for (int off = 16; off >= 1; off >>= 1) acc[j] = __fadd_rn(acc[j], __shfl_xor_sync(kFull, acc[j], off));
        }
        if (lane == 0) {
#pragma unroll
            for (int j = 0; j < kTokT; ++j) part[seg][j] = acc[j];
        }
        __syncthreads();
        if (threadIdx.x < kTokT) {
            const int t = t0 + threadIdx.x;
            if (t < T) {
                float r = part[0][threadIdx.x];
                for (int s2 = 1; s2 < nseg; ++s2) r = __fadd_rn(r, part[s2][threadIdx.x]);
                z[(size_t)t * E + e] = r;
            }
        }
        __syncthreads();
    }
}

// ---------------------------------------------------------------------------
// scores + group-limited top-k: one warp per token
// ---------------------------------------------------------------------------
__device__ __forceinline__ float canonical_sigmoid(float z) {
    const float kLog2e = 0x1.715476p+0f, kLn2Hi = 0x1.62e4p-1f, kLn2Lo = 0x1.7f7d1cp-20f;
    float a = __fsub_rn(0.0f, z);
    if (a > 87.0f) a = 87.0f;
    if (a < -87.0f) a = -87.0f;
    const float n = rintf(__fmul_rn(a, kLog2e));
    float r = __fmaf_rn(-n, kLn2Hi, a);
    r = __fmaf_rn(-n, kLn2Lo, r);
    // e^r = sum r^i / i!, i <= 7
    float p = 0x1.a01a02p-13f;
    p = __fmaf_rn(p, r, 0x1.6c16c2p-10f);
    p = __fmaf_rn(p, r, 0x1.111112p-7f);
    p = __fmaf_rn(p, r, 0x1.555556p-5f);
    p = __fmaf_rn(p, r, 0x1.555556p-3f);
    p = __fmaf_rn(p, r, 0.5f);
    p = __fmaf_rn(p, r, 1.0f);
    p = __fmaf_rn(p, r, 1.0f);
    const float two_n = __int_as_float(((int)n + 127) << 23);
    const float ex = __fmul_rn(p, two_n);
    return __fdiv_rn(1.0f, __fadd_rn(1.0f, ex));
}

// Order-preserving map of a finite fp32 value to uint32 (0 is below every
// finite value and marks "not available").
__device__ __forceinline__ uint32_t ord_key(float f) {
    const uint32_t b = __float_as_uint(f);
    return (b & 0x80000000u) ? ~b : (b | 0x80000000u);
}
// Warp argmax over one candidate per lane: largest key, then lowest index.
__device__ __forceinline__ int warp_argmax_key(uint32_t key, int idx) {
    const uint32_t kmax = __reduce_max_sync(kFull, key);
    return (int)__reduce_min_sync(kFull, key == kmax ? (uint32_t)idx : 0xffffffffu);
}

// One warp routes one token.  Lane l holds experts l, l+32, ... (E <= 256).
// uw: per-warp scratch of E floats; g_sh: per-warp scratch of G floats.
__device__ __forceinline__ void route_token(const float* __restrict__ z, const float* __restrict__ bias, int E,
                                            int G, int Gk, int K, float routed_scale, int t, float* uw,
                                            float* g_sh, int32_t* __restrict__ idx, float* __restrict__ wts) {
    const int lane = threadIdx.x & 31;
    const int gs = E / G;
    float s[8], u[8];
    int grp[8];
#pragma unroll
    for (int m = 0; m < 8; ++m) {
        const int e = lane + 32 * m;
        s[m] = 0.0f; u[m] = 0.0f; grp[m] = 0;
        if (e < E) {
            s[m] = canonical_sigmoid(z[(size_t)t * E + e]);
            u[m] = __fadd_rn(s[m], bias ? bias[e] : 0.0f);
            grp[m] = e / gs;
            uw[e] = u[m];
        }
    }
    __syncwarp();
    // group score = sum of the two largest u of the group (scan in index order)
    for (int g = lane; g < G; g += 32) {
        float top1 = -INFINITY, top2 = -INFINITY;
        const float* ug = uw + g * gs;
#pragma unroll 8
        for (int i = 0; i < gs; ++i) {
            const float v = ug[i];
            if (v > top1) { top2 = top1; top1 = v; }
            else if (v > top2) top2 = v;
        }
        g_sh[g] = gs == 1 ? top1 : __fadd_rn(top1, top2);
    }
    __syncwarp();
    // keep topk_group groups: repeated argmax, ties to the lower index
    uint64_t kept = 0;
    const uint32_t gk0 = lane < G ? ord_key(g_sh[lane]) : 0u;
    const uint32_t gk1 = lane + 32 < G ? ord_key(g_sh[lane + 32]) : 0u;
    for (int r = 0; r < Gk; ++r) {
        uint32_t k = 0u;
        int i = 0x7fffffff;
        if (lane < G && !((kept >> lane) & 1)) { k = gk0; i = lane; }
        if (lane + 32 < G && !((kept >> (lane + 32)) & 1) && gk1 > k) { k = gk1; i = lane + 32; }
        kept |= 1ull << warp_argmax_key(k, i);
    }
    // top_k experts by u among the kept groups, descending, ties to the lower id
    uint32_t key[8];
#pragma unroll
    for (int m = 0; m < 8; ++m) key[m] = (lane + 32 * m < E && ((kept >> grp[m]) & 1)) ? ord_key(u[m]) : 0u;
    int sel = 0;
    float ssum = 0.0f, mys = 0.0f;
    for (int j = 0; j < K; ++j) {
        uint32_t bk = 0u;
        int bm = 0;
#pragma unroll
        for (int m = 0; m < 8; ++m)
            if (key[m] > bk) { bk = key[m]; bm = m; }   // strict: the lower expert id wins a tie
        const int bi = warp_argmax_key(bk, lane + 32 * bm);
        float win = 0.0f;
        if ((bi & 31) == lane) {
            const int m = bi >> 5;
#pragma unroll
            for (int mm = 0; mm < 8; ++mm)
                if (mm == m) { key[mm] = 0u; win = s[mm]; }
        }
        const float sv = __shfl_sync(kFull, win, bi & 31);
        ssum = __fadd_rn(ssum, sv);   // slot order, identical on every lane
        if (lane == j) { sel = bi; mys = sv; }   // lane j keeps slot j
    }
    // weights: s_j / sum(s), summed in slot order, times routed_scale
    if (lane < K) {
        idx[(size_t)t * K + lane] = sel;
        wts[(size_t)t * K + lane] = __fmul_rn(__fdiv_rn(mys, ssum), routed_scale);
    }
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
    route_token(z, bias, d.E, d.G, d.Gk, d.K, d.routed_scale, t, u_sh[w], g_sh[w], idx, wts);
}

// ---------------------------------------------------------------------------
// permutation: one CTA; stable counting sort of entries a = t*K + j by expert
// ---------------------------------------------------------------------------
constexpr int kPermThreads = 512;
constexpr int kPermWarps = kPermThreads / 32;

// With `z` given, the same CTA first routes every token (one warp per token,
// decode-sized batches) and then permutes.  Offsets and the active list are
// kept in shared memory as well, so nothing written here is read back from
// global memory.
__global__ void __launch_bounds__(kPermThreads) permute_kernel(int32_t* __restrict__ idx, Dims d,
                                                               int32_t* __restrict__ offsets,
                                                               int32_t* __restrict__ perm,
                                                               int32_t* __restrict__ inv,
                                                               int32_t* __restrict__ active,
                                                               Plan* __restrict__ plan,
                                                               const float* __restrict__ z,
                                                               const float* __restrict__ bias,
                                                               float* __restrict__ wts) {
    const int n = d.T * d.K, E = d.E;
    __shared__ int32_t cnt[kPermWarps][kMaxExperts];   // per-warp segment counts, then cursors
    __shared__ int32_t s_off[kMaxExperts + 1];
    __shared__ int32_t s_act[kMaxExperts + 1];
    __shared__ float g_sh[kPermWarps][kMaxGroups];
    __shared__ float s_bias[kMaxExperts];
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    // the selection bias is an input no kernel of this library writes: staged
    // before the wait for the logits kernel
    if (z != nullptr)
        for (int i = threadIdx.x; i < E; i += kPermThreads) s_bias[i] = bias ? bias[i] : 0.0f;
    __syncthreads();
    pdl_wait();
    pdl_launch();
    if (z != nullptr) {
        for (int t = warp; t < d.T; t += kPermWarps)
            route_token(z, s_bias, d.E, d.G, d.Gk, d.K, d.routed_scale, t, reinterpret_cast<float*>(cnt[warp]),
                        g_sh[warp], idx, wts);
        __syncthreads();
    }
    for (int i = threadIdx.x; i < kPermWarps * kMaxExperts; i += kPermThreads) (&cnt[0][0])[i] = 0;
    __syncthreads();
    const int seg = (n + kPermWarps - 1) / kPermWarps;
    const int a0 = warp * seg, a1 = min(n, a0 + seg);
    for (int a = a0 + lane; a < a1; a += 32) atomicAdd(&cnt[warp][idx[a]], 1);
    __syncthreads();
    // per-expert totals and per-warp starting cursors (warp order = entry order)
    if (threadIdx.x < E) {
        const int e = threadIdx.x;
        int run = 0;
#pragma unroll
        for (int wv = 0; wv < kPermWarps; ++wv) { const int c = cnt[wv][e]; cnt[wv][e] = run; run += c; }
        s_off[e] = run;
    }
    __syncthreads();
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
            if (e < E) { offsets[e] = run; s_off[e] = run; }
            run += local[q];
        }
        if (lane == 31) { offsets[E] = run; s_off[E] = run; }
    }
    __syncthreads();
    for (int i = threadIdx.x; i < kPermWarps * E; i += kPermThreads) {
        const int wv = i / E, e = i - wv * E;
        cnt[wv][e] += s_off[e];
    }
    __syncthreads();
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
            inv[a] = pos;
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
            if (flags & (1 << q)) { active[1 + pos] = lane * 8 + q; s_act[1 + pos] = lane * 8 + q; ++pos; }
        if (lane == 31) { active[0] = incl; s_act[0] = incl; }
    }
    if (plan == nullptr) return;
    __syncthreads();
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

}  // namespace

cudaError_t launch_router_logits(const Dims& d, const uint16_t* x, const float* W, float* z, __half* xq, float* xs,
                                 __half* x16, uint32_t* zero_words, int n_zero, cudaStream_t s) {
    if (d.T == 0) return cudaSuccess;
    const int nseg = (d.H / 128 + 7) / 8;
    prof_begin("router_logits", s);
    cudaError_t e;
    if (xq == nullptr && d.T >= 16 && nseg <= 8) {
        // larger batches without activation preparation: tokens reused across 16 experts
        dim3 grid((d.E + kEB - 1) / kEB, (d.T + kTokT - 1) / kTokT);
        e = launch_pdl(router_logits_tile_kernel, grid, dim3(nseg * 32), 0, s, x, W, d.H, d.T, d.E, z, x16,
                       zero_words, n_zero);
    } else {
        dim3 grid(d.E, (d.T + kTok - 1) / kTok);
        e = launch_pdl(router_logits_kernel, grid, dim3(nseg * 32), 0, s, x, W, d.H, d.T, d.E, z, xq, xs, x16,
                       zero_words, n_zero);
    }
    prof_end(s);
    return e;
}

cudaError_t launch_topk(const Dims& d, const float* z, const float* bias, int32_t* idx, float* wts,
                        cudaStream_t s) {
    if (d.T == 0) return cudaSuccess;
    prof_begin("router_topk", s);
    const cudaError_t e = launch_pdl(topk_kernel, dim3((d.T + kTopkWarps - 1) / kTopkWarps), dim3(kTopkWarps * 32),
                                     0, s, z, bias, d, idx, wts);
    prof_end(s);
    return e;
}

cudaError_t launch_permute(const Dims& d, const int32_t* idx, int32_t* offsets, int32_t* perm, int32_t* inv,
                           int32_t* active, Plan* plan, cudaStream_t s) {
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
    prof_begin("route_permute", s);
    const cudaError_t e = launch_pdl(permute_kernel, dim3(1), dim3(kPermThreads), 0, s, idx, d, offsets, perm, inv,
                                     active, plan, z, bias, wts);
    prof_end(s);
    return e;
}

}  // namespace mq
