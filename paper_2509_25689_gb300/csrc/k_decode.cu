// Expert FFN kernels (decode path): SwiGLU gate/up per routed expert and
// the shared expert, then down projection with the router-weighted combine
// (arXiv 2509.25689 Fig. 1: routed experts weighted by the router plus an
// always-on shared expert).  Each tensor is dequantized in-kernel from its
// own block format.
#include "mq_internal.h"

namespace mq {
namespace {

constexpr unsigned kFull = 0xffffffffu;
constexpr int kWarps = 8;
constexpr int kTokChunk = 4;

__device__ __forceinline__ float bf16_to_f32(uint16_t v) { return __uint_as_float((uint32_t)v << 16); }
__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
    for (int off = 16; off >= 1; off >>= 1) v += __shfl_xor_sync(kFull, v, off);
    return v;
}

// grid (E + 1, I / kWarps); block slot < active count -> routed expert, slot
// E -> shared expert; one warp per intermediate row.
__global__ void __launch_bounds__(kWarps * 32) gateup_kernel(const __grid_constant__ ExpertTab tab, Dims d,
                                                            const uint16_t* __restrict__ x,
                                                            const int32_t* __restrict__ offsets,
                                                            const int32_t* __restrict__ perm,
                                                            const int32_t* __restrict__ active,
                                                            float* __restrict__ h) {
    const int slot = blockIdx.x;
    int e, n_tok, first = 0;
    const bool shared = slot == d.E;
    if (shared) {
        if (!d.has_shared) return;
        e = d.E; n_tok = d.T;
    } else {
        if (slot >= active[0]) return;
        e = active[1 + slot];
        first = offsets[e];
        n_tok = offsets[e + 1] - first;
    }
    const int lane = threadIdx.x & 31;
    const int r = blockIdx.y * kWarps + (threadIdx.x >> 5);
    if (r >= d.I) return;
    const int fg = tab.fmt[e][0], fu = tab.fmt[e][1];
    const uint8_t* pg = tab.p[e][0];
    const uint8_t* pu = tab.p[e][1];
    const TensorLayout Lg = tensor_layout(fg, d.I, d.H), Lu = tensor_layout(fu, d.I, d.H);
    for (int c0 = 0; c0 < n_tok; c0 += kTokChunk) {
        int a[kTokChunk], tk[kTokChunk];
        float g[kTokChunk], u[kTokChunk];
#pragma unroll
        for (int j = 0; j < kTokChunk; ++j) {
            const int q = c0 + j;
            a[j] = -1; tk[j] = 0; g[j] = 0.0f; u[j] = 0.0f;
            if (q < n_tok) {
                if (shared) { tk[j] = q; a[j] = d.T * d.K + q; }
                else { a[j] = perm[first + q]; tk[j] = a[j] / d.K; }
            }
        }
        for (int k = lane; k < d.H; k += 32) {
            const float wg = dequant_at(fg, pg, Lg, r, k);
            const float wu = dequant_at(fu, pu, Lu, r, k);
#pragma unroll
            for (int j = 0; j < kTokChunk; ++j) {
                if (a[j] >= 0) {
                    const float xv = bf16_to_f32(x[(size_t)tk[j] * d.H + k]);
                    g[j] = fmaf(wg, xv, g[j]);
                    u[j] = fmaf(wu, xv, u[j]);
                }
            }
        }
#pragma unroll
        for (int j = 0; j < kTokChunk; ++j) {
            const float gs = warp_sum(g[j]), us = warp_sum(u[j]);
            if (lane == 0 && a[j] >= 0) h[(size_t)a[j] * d.I + r] = gs / (1.0f + expf(-gs)) * us;
        }
    }
}

// grid H / kWarps; one warp per output row; combine in slot order, then the
// shared expert.
__global__ void __launch_bounds__(kWarps * 32) down_kernel(const __grid_constant__ ExpertTab tab, Dims d,
                                                          const int32_t* __restrict__ idx,
                                                          const float* __restrict__ wts,
                                                          const float* __restrict__ h, float* __restrict__ out) {
    const int lane = threadIdx.x & 31;
    const int r = blockIdx.x * kWarps + (threadIdx.x >> 5);
    if (r >= d.H) return;
    for (int t = 0; t < d.T; ++t) {
        float y = 0.0f;
        for (int j = 0; j < d.K + d.has_shared; ++j) {
            const bool sh = j == d.K;
            const int a = sh ? d.T * d.K + t : t * d.K + j;
            const int e = sh ? d.E : idx[a];
            const int f = tab.fmt[e][2];
            const uint8_t* p = tab.p[e][2];
            const TensorLayout L = tensor_layout(f, d.H, d.I);
            float acc = 0.0f;
            for (int i = lane; i < d.I; i += 32) acc = fmaf(dequant_at(f, p, L, r, i), h[(size_t)a * d.I + i], acc);
            acc = warp_sum(acc);
            y = sh ? y + acc : fmaf(wts[a], acc, y);
        }
        if (lane == 0) out[(size_t)t * d.H + r] = y;
    }
}

}  // namespace

cudaError_t launch_decode_ffn(const Dims& d, const ExpertTab& tab, const uint16_t* x, const Work& w, float* out,
                              cudaStream_t s) {
    if (d.T == 0) return cudaSuccess;
    dim3 g1(d.E + 1, (d.I + kWarps - 1) / kWarps);
    prof_begin("gateup", s);
    gateup_kernel<<<g1, kWarps * 32, 0, s>>>(tab, d, x, w.offsets, w.perm, w.active, w.h);
    prof_end(s);
    cudaError_t err = cudaGetLastError();
    if (err != cudaSuccess) return err;
    prof_begin("down", s);
    down_kernel<<<(d.H + kWarps - 1) / kWarps, kWarps * 32, 0, s>>>(tab, d, w.idx, w.wts, w.h, out);
    prof_end(s);
    return cudaGetLastError();
}

}  // namespace mq
