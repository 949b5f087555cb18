// Activation preparation for the tensor-core GEMV kernels.
//
// The decode kernels multiply packed weight codes (MMA operand A) by an
// activation vector (operand B).  Operand A is one masked code word read as
// fp16x2: the code bits land in the mantissa of an fp16 subnormal, so a
// code c at bit offset s of its 16-bit half reads as c * 2^(s - 24), exact
// (the tensor cores take fp16 subnormals as they are).  For every activation
// vector (a token's hidden state, or a SwiGLU output) this prepares, per
// 32-element block:
//   - sigma = 2^ex, ex chosen so the block maximum scales into [2^12, 2^13);
//     xt = fp16(v / sigma) is the fp16 activation every kernel uses (exact
//     for bf16 inputs), and c = 2^24 * sigma undoes both scalings;
//   - fp16 copies of xt in natural element order, one per code family, each
//     element divided by the power of two its code carries: F2 (2-bit code
//     positions: Q2_K, and Q3_K whose high bit the kernels place right above
//     the pair's 2-bit code), F4 (4-bit codes: Q4_K, and Q6_K whose high two
//     bits the kernels weigh through shifts and exact operand scalings), F8
//     (8-bit codes: Q8_0, none);
//   - for bf16 weights (MMA operands of one type: bf16 x bf16), the value
//     itself split into bf16 hi = bf16(v) and lo = bf16(v - hi) (hi + lo
//     holds v to about 16 bits; for a bf16 token lo is 0), each in the
//     tensor-core fragment order of the BF16 weight blocks (families FB and
//     FBL);
//   - the sums sigma * sum(xt) over every 16- and 32-element sub-block (the
//     sub-block min terms of Q2_K / Q4_K, the -4 offset of Q3_K codes and the
//     +128 offset of Q8_0 codes).
// Layout per vector: halves [kFamSlots family slots][nsb][256] and, per
// superblock, a 32-float record {c[8] | S16[16] in slot order | S32[8]}.
#pragma once
#include <cuda_bf16.h>
#include <cuda_fp16.h>
#include <stdint.h>

#include "mq_layout.h"

namespace mq {

enum Family : int { kF2 = 0, kFB = 1, kF4 = 2, kF8 = 3, kFBL = 4 };
constexpr int kFamSlots = 5;
// families every prepared token gets (the bf16 pair only when a gate or up
// tensor of the layer is BF16)
constexpr int kCodeFams = (1 << kF2) | (1 << kF4) | (1 << kF8);
constexpr int kBf16Fams = (1 << kFB) | (1 << kFBL);

constexpr int kStatFloats = 32;   // floats of statistics per superblock
constexpr int kStatC = 0, kStatS16 = 8, kStatS32 = 24;

// power of two carried by the code pair m of each family (bit offset of the
// code inside its fp16 half after the word is read, see the decode kernels)
__host__ __device__ __forceinline__ int pair_shift2(int m) { return m <= 4 ? 2 * m : 2 * (m - 5); }   // m < 8
__host__ __device__ __forceinline__ int pair_shift4(int m) { return 4 * (m & 1); }                    // m < 16

// slot of 16-wide sub-block j (< 16): lane t of a warp owns slots 4t..4t+3,
// i.e. sub-blocks 2t, 2t+1, 8+2t, 9+2t
__host__ __device__ __forceinline__ int slot16(int j) { return 4 * ((j & 7) >> 1) + 2 * (j >> 3) + (j & 1); }

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
    const int s = jb >> 3, kk = ((jb & 7) << 5) + lane;                // element of superblock s
    __half* qs = q + (size_t)s * 256 + kk;
    const size_t fam_stride = (size_t)nsb * 256;
    const int m16 = (kk & 15) >> 1, m32 = (kk & 31) >> 1;
    if (fam_mask & (1 << kF2)) qs[kF2 * fam_stride] = __float2half_rn(ldexpf(xt, -pair_shift2(m16)));
    if (fam_mask & (1 << kF4)) qs[kF4 * fam_stride] = __float2half_rn(ldexpf(xt, -pair_shift4(m32)));
    if (fam_mask & (1 << kF8)) qs[kF8 * fam_stride] = __float2half_rn(xt);
    if (fam_mask & (1 << kFB)) {
        const __nv_bfloat16 hi = __float2bfloat16_rn(v);
        const __nv_bfloat16 lo = __float2bfloat16_rn(v - __bfloat162float(hi));   // v - hi is exact
        unsigned short* fb = reinterpret_cast<unsigned short*>(q + (size_t)s * 256 + ((jb & 7) << 5) + bf16_slot(lane));
        fb[kFB * fam_stride] = __bfloat16_as_ushort(hi);
        fb[kFBL * fam_stride] = __bfloat16_as_ushort(lo);
    }
    const float s16 = half_warp_sum(xt);
    const float s32 = s16 + __shfl_xor_sync(0xffffffffu, s16, 16);
    float* rec = st + (size_t)s * kStatFloats;
    if ((lane & 15) == 0) {
        const int j = ((jb & 7) << 1) + (lane >> 4);   // 16-wide sub-block in the superblock
        rec[kStatS16 + slot16(j)] = s16 * sigma;
    }
    if (lane == 0) {
        rec[kStatC + (jb & 7)] = 16777216.0f * sigma;
        rec[kStatS32 + (jb & 7)] = s32 * sigma;
    }
}

// family mask needed by a weight format
__host__ __device__ __forceinline__ int families_of(int fmt) {
    return fmt == kQ2K || fmt == kQ3K ? (1 << kF2)
         : fmt == kQ4K || fmt == kQ6K ? (1 << kF4)
         : fmt == kBF16 ? kBf16Fams : (1 << kF8);
}

}  // namespace mq
