// Expert selection for one token by one warp (arXiv 2509.25689 Sec. 3.2:
// sigmoid expert scores plus the selection bias, topk_group groups ranked by
// the sum of their two best scores, then num_experts_per_tok experts from
// the kept groups; weights are the selected sigmoid scores normalised in slot
// order and scaled by routed_scale).  Canonical fp32 order, so ids and
// weights are bit-exact with the CPU reference:
//   sigmoid: Cody-Waite reduction a = n ln2 + r, degree-7 Taylor for e^r
//            (coefficients 1/i! rounded to fp32, Horner), exact 2^n scaling,
//            1/(1+e) with IEEE division; |a| clamped to 87.
//   select:  ties go to the lower group / expert index.
// Used by the routing kernels and by the one-token FFN kernels, which route
// their token themselves.
#pragma once
#include <cuda_runtime.h>
#include <stdint.h>

namespace mq {
namespace sel {

constexpr unsigned kFull = 0xffffffffu;

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
                                            float* g_sh, int32_t* __restrict__ idx, float* __restrict__ wts,
                                            int* sel_out = nullptr) {
    const int lane = threadIdx.x & 31;
    const int gs = E / G;
    float s[8], u[8];
    int grp[8];
#pragma unroll
    for (int m = 0; m < 8; ++m) {
        const int e = lane + 32 * m;
        s[m] = 0.0f; u[m] = 0.0f; grp[m] = 0;
        if (e < E) {
            // through L2: the logits may come from other CTAs of the same grid
            s[m] = canonical_sigmoid(__ldcg(z + (size_t)t * E + e));
            u[m] = __fadd_rn(s[m], bias ? bias[e] : 0.0f);
            grp[m] = e / gs;
            uw[e] = u[m];
        }
    }
    __syncwarp();
    // group score = sum of the two largest u of the group.  P lanes share a
    // group (P * G <= 32): each keeps the two largest of a strided part, then
    // the pairs are merged over the P lanes (the two largest of a set do not
    // depend on the order they are found in).
    if (G <= 16) {
        int P = 2;
        while (P * 2 * G <= 32) P *= 2;
        const int g = lane / P, sub = lane % P;
        float top1 = -INFINITY, top2 = -INFINITY;
        if (g < G) {
            const float* ug = uw + g * gs;
            for (int i = sub; i < gs; i += P) {
                const float v = ug[i];
                top2 = fmaxf(top2, fminf(top1, v));
                top1 = fmaxf(top1, v);
            }
        }
        for (int off = P >> 1; off >= 1; off >>= 1) {
            const float o1 = __shfl_xor_sync(kFull, top1, off), o2 = __shfl_xor_sync(kFull, top2, off);
            top2 = fmaxf(fminf(top1, o1), fmaxf(top2, o2));
            top1 = fmaxf(top1, o1);
        }
        if (g < G && sub == 0) g_sh[g] = gs == 1 ? top1 : __fadd_rn(top1, top2);
    } else {
        for (int g = lane; g < G; g += 32) {
            float top1 = -INFINITY, top2 = -INFINITY;
            const float* ug = uw + g * gs;
            for (int i = 0; i < gs; ++i) {
                const float v = ug[i];
                top2 = fmaxf(top2, fminf(top1, v));
                top1 = fmaxf(top1, v);
            }
            g_sh[g] = gs == 1 ? top1 : __fadd_rn(top1, top2);
        }
    }
    __syncwarp();
    // keep the topk_group best groups (largest score, ties to the lower
    // index): group g is kept when fewer than topk_group groups come before it
    uint64_t kept = 0;
#pragma unroll
    for (int h = 0; h < 2; ++h) {
        const int g = lane + 32 * h;
        bool keep = false;
        if (g < G) {
            const uint32_t kg = ord_key(g_sh[g]);
            int before = 0;
            for (int g2 = 0; g2 < G; ++g2) {
                const uint32_t k2 = ord_key(g_sh[g2]);
                before += (k2 > kg || (k2 == kg && g2 < g)) ? 1 : 0;
            }
            keep = before < Gk;
        }
        kept |= (uint64_t)__ballot_sync(kFull, keep) << (32 * h);
    }
    // the scores s replace u in the scratch (u stays in registers)
    __syncwarp();
#pragma unroll
    for (int m = 0; m < 8; ++m)
        if (lane + 32 * m < E) uw[lane + 32 * m] = s[m];
    // top_k experts by u among the kept groups, descending, ties to the lower
    // id: each lane orders its candidates once, then every round takes the
    // best head over the warp and the winning lane drops its head
    uint32_t key[8];
    int id[8];
#pragma unroll
    for (int m = 0; m < 8; ++m) {
        key[m] = (lane + 32 * m < E && ((kept >> grp[m]) & 1)) ? ord_key(u[m]) : 0u;
        id[m] = lane + 32 * m;
    }
    auto cmpx = [&](int a, int b) {   // position a before b: larger key, then lower id
        const bool sw = key[b] > key[a] || (key[b] == key[a] && id[b] < id[a]);
        const uint32_t ka = key[a], kb = key[b];
        const int ia = id[a], ib = id[b];
        key[a] = sw ? kb : ka; key[b] = sw ? ka : kb;
        id[a] = sw ? ib : ia; id[b] = sw ? ia : ib;
    };
    cmpx(0, 1); cmpx(2, 3); cmpx(4, 5); cmpx(6, 7);
    cmpx(0, 2); cmpx(1, 3); cmpx(4, 6); cmpx(5, 7);
    cmpx(1, 2); cmpx(5, 6);
    cmpx(0, 4); cmpx(1, 5); cmpx(2, 6); cmpx(3, 7);
    cmpx(2, 4); cmpx(3, 5);
    cmpx(1, 2); cmpx(3, 4); cmpx(5, 6);
    __syncwarp();
    int sel = 0;
    float ssum = 0.0f, mys = 0.0f;
    for (int j = 0; j < K; ++j) {
        const uint32_t kmax = __reduce_max_sync(kFull, key[0]);
        const int bi = (int)__reduce_min_sync(kFull, key[0] == kmax ? (uint32_t)id[0] : 0xffffffffu);
        if ((bi & 31) == lane) {
#pragma unroll
            for (int m = 0; m < 7; ++m) { key[m] = key[m + 1]; id[m] = id[m + 1]; }
            key[7] = 0u; id[7] = 0x7fffffff;
        }
        const float sv = uw[bi];
        ssum = __fadd_rn(ssum, sv);   // slot order, identical on every lane
        if (lane == j) { sel = bi; mys = sv; }   // lane j keeps slot j
    }
    // weights: s_j / sum(s), summed in slot order, times routed_scale
    if (lane < K) {
        idx[(size_t)t * K + lane] = sel;
        wts[(size_t)t * K + lane] = __fmul_rn(__fdiv_rn(mys, ssum), routed_scale);
    }
    if (sel_out != nullptr) *sel_out = sel;
}


// The same selection for one token, written for a cold SM: it runs once per
// decode call in whichever CTA routes, where every distinct line of
// instructions costs an instruction fetch from the memory system.  So the
// per-expert work is a loop (not unrolled), and the top-k is K rounds of a
// warp-wide "largest key, then lowest id" over each lane's 8 candidates
// (equal to route_token's per-lane ordering plus head merge).  Scratch:
// sc[2 * kMaxExperts] floats (u, then s), g_sh[G].  Results are identical to
// route_token's.
__device__ __forceinline__ void route_token_compact(const float* __restrict__ z, const float* __restrict__ bias,
                                                    int E, int G, int Gk, int K, float routed_scale, int t,
                                                    float* sc, float* g_sh, int32_t* __restrict__ idx,
                                                    float* __restrict__ wts, int* sel_out) {
    const int lane = threadIdx.x & 31;
    const int gs = E / G;
    float* u_sh = sc;
    float* s_sh = sc + 256;
    // the token's logits (E <= 256: at most 8 per lane) as one batch of
    // independent loads, then the scores in a rolled loop (small code)
    float zv[8];
#pragma unroll
    for (int m = 0; m < 8; ++m) {
        const int e = lane + 32 * m;
        zv[m] = e < E ? __ldcg(z + (size_t)t * E + e) : 0.0f;
    }
#pragma unroll 1
    for (int m = 0; 32 * m < E; ++m) {
        const int e = lane + 32 * m;
        float zm = zv[0];
#pragma unroll
        for (int q = 1; q < 8; ++q) zm = q == m ? zv[q] : zm;
        if (e < E) {
            const float sv = canonical_sigmoid(zm);
            s_sh[e] = sv;
            u_sh[e] = __fadd_rn(sv, bias ? bias[e] : 0.0f);
        }
    }
    __syncwarp();
    // group score = sum of the two largest u of the group (as route_token)
    if (G <= 16) {
        int P = 2;
        while (P * 2 * G <= 32) P *= 2;
        const int g = lane / P, sub = lane % P;
        float top1 = -INFINITY, top2 = -INFINITY;
        if (g < G) {
            const float* ug = u_sh + g * gs;
#pragma unroll 1
            for (int i = sub; i < gs; i += P) {
                const float v = ug[i];
                top2 = fmaxf(top2, fminf(top1, v));
                top1 = fmaxf(top1, v);
            }
        }
#pragma unroll 1
        for (int off = P >> 1; off >= 1; off >>= 1) {
            const float o1 = __shfl_xor_sync(kFull, top1, off), o2 = __shfl_xor_sync(kFull, top2, off);
            top2 = fmaxf(fminf(top1, o1), fmaxf(top2, o2));
            top1 = fmaxf(top1, o1);
        }
        if (g < G && sub == 0) g_sh[g] = gs == 1 ? top1 : __fadd_rn(top1, top2);
    } else {
#pragma unroll 1
        for (int g = lane; g < G; g += 32) {
            float top1 = -INFINITY, top2 = -INFINITY;
            const float* ug = u_sh + g * gs;
#pragma unroll 1
            for (int i = 0; i < gs; ++i) {
                const float v = ug[i];
                top2 = fmaxf(top2, fminf(top1, v));
                top1 = fmaxf(top1, v);
            }
            g_sh[g] = gs == 1 ? top1 : __fadd_rn(top1, top2);
        }
    }
    __syncwarp();
    // kept groups: fewer than topk_group groups rank before them
    uint64_t kept = 0;
#pragma unroll 1
    for (int h = 0; h < 2; ++h) {
        const int g = lane + 32 * h;
        bool keep = false;
        if (g < G) {
            const uint32_t kg = ord_key(g_sh[g]);
            int before = 0;
#pragma unroll 1
            for (int g2 = 0; g2 < G; ++g2) {
                const uint32_t k2 = ord_key(g_sh[g2]);
                before += (k2 > kg || (k2 == kg && g2 < g)) ? 1 : 0;
            }
            keep = before < Gk;
        }
        kept |= (uint64_t)__ballot_sync(kFull, keep) << (32 * h);
    }
    uint32_t key[8];
#pragma unroll
    for (int m = 0; m < 8; ++m) {
        const int e = lane + 32 * m;
        key[m] = (e < E && ((kept >> (e / gs)) & 1)) ? ord_key(u_sh[e]) : 0u;
    }
    int sel = 0;
    float ssum = 0.0f, mys = 0.0f;
#pragma unroll 1
    for (int j = 0; j < K; ++j) {
        // this lane's best: largest key, the lower id first among equal keys
        uint32_t bk = 0u;
        int bm = 0;
#pragma unroll
        for (int m = 0; m < 8; ++m)
            if (key[m] > bk) { bk = key[m]; bm = m; }
        const uint32_t kmax = __reduce_max_sync(kFull, bk);
        const int bi = (int)__reduce_min_sync(kFull, bk == kmax ? (uint32_t)(lane + 32 * bm) : 0xffffffffu);
        if ((bi & 31) == lane) {
#pragma unroll
            for (int m = 0; m < 8; ++m)
                if (m == (bi >> 5)) key[m] = 0u;
        }
        const float sv = s_sh[bi];
        ssum = __fadd_rn(ssum, sv);   // slot order, identical on every lane
        if (lane == j) { sel = bi; mys = sv; }
    }
    if (lane < K) {
        idx[(size_t)t * K + lane] = sel;
        wts[(size_t)t * K + lane] = __fmul_rn(__fdiv_rn(mys, ssum), routed_scale);
    }
    if (sel_out != nullptr) *sel_out = sel;
}

}  // namespace sel
}  // namespace mq
