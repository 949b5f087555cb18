// Activation preparation for the tensor-core GEMV kernels.
//
// The decode kernels multiply packed weight codes (MMA operand A, built as
// fp16 "1024 + s*q" with a positional power-of-two s) by an activation
// vector (operand B).  For every activation vector (a token's hidden state,
// or a SwiGLU output) this prepares, per 32-element block:
//   - sigma = 2^ex, ex chosen so the block maximum scales into [2^12, 2^13)
//     (headroom for the x4 of the Q3_K high-bit family within fp16 range);
//     xt = fp16(v / sigma) is the fp16 activation every kernel uses;
//   - four fp16 copies of xt in MMA-fragment order, one per code family,
//     each element divided by the positional scale its code will carry:
//       F2 (2-bit codes: Q2_K, low bits of Q3_K), F1 (Q3_K high bit, times 4),
//       F4 (4-bit codes: Q4_K), F8 (8-bit codes: Q8_0);
//   - sums that remove the constant offset of the codes (1024, or 1152 for
//     Q8_0) and supply the sub-block min terms, already multiplied by sigma.
// Layout per vector: halves [4 families][nsb][256] and floats [80 * nsb].
#pragma once
#include <cuda_fp16.h>
#include <stdint.h>

namespace mq {

enum Family : int { kF2 = 0, kF1 = 1, kF4 = 2, kF8 = 3 };

// float offsets inside a vector's statistics record (nsb superblocks)
struct StatOff {
    int sig, os2, oq3, sxs16, os4, sxs32, os8, total;
};
__host__ __device__ __forceinline__ StatOff stat_off(int nsb) {
    StatOff o;
    o.sig = 0; o.os2 = 8 * nsb; o.oq3 = 24 * nsb; o.sxs16 = 40 * nsb;
    o.os4 = 56 * nsb; o.sxs32 = 64 * nsb; o.os8 = 72 * nsb; o.total = 80 * nsb;
    return o;
}

// positional scale of a 2-bit code pair at position p (0..7) of its word:
// p <= 4 read in place (4^p), p >= 5 read after a 10-bit shift (4^(p-5))
__host__ __device__ __forceinline__ int pos_shift2(int p) { return p <= 4 ? 2 * p : 2 * (p - 5); }
// high-bit plane: pair position p1 (0..15): in place up to 9, then shifted by 10
__host__ __device__ __forceinline__ int pos_shift1(int p1) { return p1 <= 9 ? p1 : p1 - 10; }

// index of element kk (0..255 in a superblock) inside the fragment block:
// thread (g, t4) of a warp reads 8 consecutive halves at (g*4 + t4)*8.
__device__ __forceinline__ int frag_index(bool wide32, int kk) {
    const int i = kk >> 4, r = kk & 15;
    const int h = r >> 3, t4 = (r & 7) >> 1, e = r & 1;
    const int g = wide32 ? (i >> 1) : (i & 7);
    const int sel = wide32 ? (i & 1) : (i >> 3);
    return (g * 4 + t4) * 8 + sel * 4 + h * 2 + e;
}

__device__ __forceinline__ float warp_max_abs(float v) {
    v = fabsf(v);
#pragma unroll
    for (int off = 16; off >= 1; off >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, off));
    return v;
}
__device__ __forceinline__ float half_warp_sum(float v) {
#pragma unroll
    for (int off = 8; off >= 1; off >>= 1) v += __shfl_xor_sync(0xffffffffu, v, off);
    return v;
}

// Warp-cooperative: lane l holds element v = vec[32*jb + l] (0 past the end).
// fam_mask: bit f set -> write family f.  q: halves [4][nsb*256]; st: stats.
__device__ __forceinline__ void prep_block32(float v, int jb, int fam_mask, __half* __restrict__ q,
                                             float* __restrict__ st, int nsb) {
    const int lane = threadIdx.x & 31;
    const float amax = warp_max_abs(v);
    int ex = 0;
    if (amax > 0.0f) ex = ilogbf(amax) - 12;
    const float inv_sigma = ldexpf(1.0f, -ex), sigma = ldexpf(1.0f, ex);
    const float xt = __half2float(__float2half_rn(v * inv_sigma));   // the fp16 activation
    const int s = jb >> 3, kk = ((jb & 7) << 5) + lane;
    const int i = kk >> 4, r = kk & 15, h = r >> 3;
    __half* qs = q + (size_t)s * 256;
    const size_t fam_stride = (size_t)nsb * 256;
    const int p2 = 2 * (i & 3) + h;
    const float x2 = ldexpf(xt, -pos_shift2(p2));
    const int p1 = 2 * (i & 7) + h;
    const float x1 = ldexpf(4.0f * xt, -pos_shift1(p1));
    const float x4 = h ? xt * 0.0625f : xt;
    if (fam_mask & (1 << kF2)) qs[kF2 * fam_stride + frag_index(false, kk)] = __float2half_rn(x2);
    if (fam_mask & (1 << kF1)) qs[kF1 * fam_stride + frag_index(false, kk)] = __float2half_rn(x1);
    if (fam_mask & (1 << kF4)) qs[kF4 * fam_stride + frag_index(true, kk)] = __float2half_rn(x4);
    if (fam_mask & (1 << kF8)) qs[kF8 * fam_stride + frag_index(true, kk)] = __float2half_rn(xt);
    // sums use exactly the fp16 values the MMA sees
    const float sx16 = half_warp_sum(xt);
    const float o2 = 1024.0f * half_warp_sum(__half2float(__float2half_rn(x2)));
    const float o1 = 1024.0f * half_warp_sum(__half2float(__float2half_rn(x1)));
    const float o4h = 1024.0f * half_warp_sum(__half2float(__float2half_rn(x4)));
    const float o8h = 1152.0f * half_warp_sum(xt);   // Q8_0 codes read as 1024 + (q + 128)
    const float sx32 = sx16 + __shfl_xor_sync(0xffffffffu, sx16, 16);
    const float o4 = o4h + __shfl_xor_sync(0xffffffffu, o4h, 16);
    const float o8 = o8h + __shfl_xor_sync(0xffffffffu, o8h, 16);
    const StatOff so = stat_off(nsb);
    if ((lane & 15) == 0) {
        const int jj = ((jb & 7) << 1) + (lane >> 4);          // 16-wide sub-block in the superblock
        const int tile = jj >> 3, n = jj & 7;
        const int idx = s * 16 + (n >> 1) * 4 + tile * 2 + (n & 1);
        st[so.os2 + idx] = o2 * sigma;
        st[so.sxs16 + idx] = sx16 * sigma;
        st[so.oq3 + idx] = (o2 + o1) * sigma + 4.0f * sx16 * sigma;
    }
    if (lane == 0) {
        st[so.sig + jb] = sigma;
        st[so.os4 + jb] = o4 * sigma;
        st[so.sxs32 + jb] = sx32 * sigma;
        st[so.os8 + jb] = o8 * sigma;
    }
}

// family mask needed by a weight format
__host__ __device__ __forceinline__ int families_of(int fmt) {
    return fmt == 1 ? (1 << kF2) : fmt == 2 ? ((1 << kF2) | (1 << kF1)) : fmt == 3 ? (1 << kF4) : (1 << kF8);
}

}  // namespace mq
