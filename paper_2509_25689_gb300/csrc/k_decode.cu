// Expert FFN kernels for decode-sized batches (arXiv 2509.25689 Fig. 1: a
// shared expert plus router-weighted routed SwiGLU experts; each expert
// tensor stored in its own k-quant style block format, Sec. 3.3).
//
// Dequant-fused GEMV on the legacy tensor-core path (mma.sync m16n8k16,
// fp16 x fp16 -> fp32):
//   A (16 rows x 16 k) = weight codes as fp16 "1024 + s*q" built with one
//     LOP3 per code pair straight from the packed words (s = a positional
//     power of two, so most pairs need no shift);
//   B (16 k x 8 cols) = the prepared activation (mq_actprep.cuh), column n
//     carrying sub-block n of the 256-weight superblock and zero elsewhere;
//   D (16 rows x 8 cols) = per-(row, sub-block) partial dot products, so the
//     sub-block scales and mins are applied once per 16x256 tile in fp32.
// Work is cut into warp items (32 rows x a K range of one tensor of one
// expert) taken from a global counter; partial sums go to scratch and the
// last warp to finish a row block combines them in a fixed order (SwiGLU for
// gate/up, routed + shared sum for down), so results are deterministic.
#include <cuda_fp16.h>

#include "mq_actprep.cuh"
#include "mq_internal.h"

namespace mq {
namespace {

constexpr unsigned kFull = 0xffffffffu;
constexpr int kWarpsPerCta = 8;
constexpr int kMaxSplit = 4;

__device__ __forceinline__ uint32_t lop3_and_or(uint32_t a, uint32_t mask, uint32_t orv) {
    uint32_t d;
    asm("lop3.b32 %0, %1, %2, %3, 0xEA;" : "=r"(d) : "r"(a), "r"(mask), "r"(orv));   // (a & b) | c
    return d;
}
// Q8_0: byte u -> fp16 1024 + (u ^ 0x80) in each half: M ? (a ^ K) : K
__device__ __forceinline__ uint32_t lop3_q8(uint32_t a) {
    uint32_t d;
    asm("lop3.b32 %0, %1, %2, %3, 0x6A;" : "=r"(d) : "r"(a), "r"(0x00FF00FFu), "r"(0x64806480u));
    return d;
}
__device__ __forceinline__ uint32_t hmul2u(uint32_t a, uint32_t b) {
    __half2 x = *reinterpret_cast<__half2*>(&a), y = *reinterpret_cast<__half2*>(&b);
    __half2 z = __hmul2(x, y);
    return *reinterpret_cast<uint32_t*>(&z);
}
__device__ __forceinline__ void mma16816(float (&d)[4], uint32_t a0, uint32_t a1, uint32_t a2, uint32_t a3,
                                         uint32_t b0, uint32_t b1) {
    asm("mma.sync.aligned.m16n8k16.row.col.f32.f16.f16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, {%0,%1,%2,%3};"
        : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
        : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1));
}

__device__ __forceinline__ uint4 ldg128(const void* p) { return __ldg(reinterpret_cast<const uint4*>(p)); }
__device__ __forceinline__ uint2 ldg64(const void* p) { return __ldg(reinterpret_cast<const uint2*>(p)); }
__device__ __forceinline__ uint32_t ldg32(const void* p) { return __ldg(reinterpret_cast<const unsigned int*>(p)); }
__device__ __forceinline__ uint32_t ldg16(const void* p) { return __ldg(reinterpret_cast<const unsigned short*>(p)); }
__device__ __forceinline__ float h2f(uint32_t bits16) { return __half2float(__ushort_as_half((unsigned short)bits16)); }

// 2-bit code pair at position p of word w as fp16x2 "1024 + 4^pos q"
template <int P>
__device__ __forceinline__ uint32_t ext2(uint32_t w, uint32_t w10) {
    constexpr int pos = P <= 4 ? P : P - 5;
    return lop3_and_or(P <= 4 ? w : w10, 0x00030003u << (2 * pos), 0x64006400u);
}
template <int P1>
__device__ __forceinline__ uint32_t ext1(uint32_t w, uint32_t w10) {
    constexpr int pos = P1 <= 9 ? P1 : P1 - 10;
    return lop3_and_or(P1 <= 9 ? w : w10, 0x00010001u << pos, 0x64006400u);
}

struct VecSrc {
    const __half* q;     // prepared fp16 fragments of vector 0
    const float* st;     // statistics of vector 0
    size_t q_stride;     // halves between vectors
    size_t st_stride;    // floats between vectors
    int nsb;             // superblocks along the contraction
};

// Per-warp GEMV on one item: rows [row0, row0+32) of a packed tensor, superblocks
// [sb0, sb1), NT activation vectors.  acc[t][tile][h]: row row0 + 16*tile + g + 8*h
// partial over this lane's sub-block slots.  Each code fragment is extracted
// once per superblock and multiplied with every vector.
template <int FMT, int NT>
__device__ __forceinline__ void gemv_item(const uint8_t* __restrict__ base, const TensorLayout& L, int row0,
                                          int sb0, int sb1, const int (&vec)[NT], const VecSrc& vs,
                                          float (&acc)[NT][2][2]) {
    const int lane = threadIdx.x & 31, g = lane >> 2, t4 = lane & 3;
    uint32_t mask[8];
#pragma unroll
    for (int n = 0; n < 8; ++n) mask[n] = (g == n) ? 0x3C003C00u : 0u;
    constexpr bool kWide = FMT == kQ4K || FMT == kQ80;
    constexpr int kTiles = kWide ? 1 : 2;
    constexpr int kFam = FMT == kQ2K || FMT == kQ3K ? kF2 : FMT == kQ4K ? kF4 : kF8;
    constexpr int kWords = FMT == kQ4K ? 8 : 4;
    const StatOff so = stat_off(vs.nsb);
    const size_t fam_stride = (size_t)vs.nsb * 256;
    int64_t rowblk[2][2];
#pragma unroll
    for (int rt = 0; rt < 2; ++rt)
#pragma unroll
        for (int hl = 0; hl < 2; ++hl) rowblk[rt][hl] = (int64_t)(row0 + 16 * rt + 8 * hl + g) * L.blocks_per_row;

    for (int s = sb0; s < sb1; ++s) {
        // ---- this lane's codes and fields for rows g, g+8 of both tiles
        uint32_t cw[2][2][kWords];
        uint32_t hw[2][2][2];
        uint32_t fld[2][2];
        float dd[2][2], dm[2][2];
#pragma unroll
        for (int rt = 0; rt < 2; ++rt) {
#pragma unroll
            for (int hl = 0; hl < 2; ++hl) {
                if (FMT == kQ80) {
                    const int64_t b0 = rowblk[rt][hl] + 8 * (int64_t)s;
                    uint32_t dv = 0;
                    if (8 * s + 2 * t4 < L.blocks_per_row) dv = ldg32(base + L.plane[0] + (b0 + 2 * t4) * 2);
                    dd[rt][hl] = h2f(dv & 0xffffu);   // block 2*t4
                    dm[rt][hl] = h2f(dv >> 16);       // block 2*t4 + 1
                } else {
                    const int64_t blk = rowblk[rt][hl] + s;
                    if (FMT == kQ2K) {
                        const uint4 v = ldg128(base + L.plane[3] + blk * 64 + 16 * t4);
                        cw[rt][hl][0] = v.x; cw[rt][hl][1] = v.y; cw[rt][hl][2] = v.z; cw[rt][hl][3] = v.w;
                        fld[rt][hl] = ldg32(base + L.plane[2] + blk * 16 + 4 * t4);
                        dd[rt][hl] = h2f(ldg16(base + L.plane[0] + blk * 2));
                        dm[rt][hl] = h2f(ldg16(base + L.plane[1] + blk * 2));
                    } else if (FMT == kQ3K) {
                        const uint4 v = ldg128(base + L.plane[2] + blk * 64 + 16 * t4);
                        cw[rt][hl][0] = v.x; cw[rt][hl][1] = v.y; cw[rt][hl][2] = v.z; cw[rt][hl][3] = v.w;
                        const uint2 hv = ldg64(base + L.plane[3] + blk * 32 + 8 * t4);
                        hw[rt][hl][0] = hv.x; hw[rt][hl][1] = hv.y;
                        const uint8_t* sp = base + L.plane[1] + blk * 12;
                        fld[rt][hl] = ldg16(sp + 2 * t4) | ((uint32_t)__ldg(sp + 8 + t4) << 16);
                        dd[rt][hl] = h2f(ldg16(base + L.plane[0] + blk * 2));
                    } else {  // Q4_K
                        const uint4 v0 = ldg128(base + L.plane[3] + blk * 128 + 32 * t4);
                        const uint4 v1 = ldg128(base + L.plane[3] + blk * 128 + 32 * t4 + 16);
                        cw[rt][hl][0] = v0.x; cw[rt][hl][1] = v0.y; cw[rt][hl][2] = v0.z; cw[rt][hl][3] = v0.w;
                        cw[rt][hl][4] = v1.x; cw[rt][hl][5] = v1.y; cw[rt][hl][6] = v1.z; cw[rt][hl][7] = v1.w;
                        const uint8_t* sp = base + L.plane[2] + blk * 12;
                        fld[rt][hl] = ldg16(sp + 2 * t4) | ((uint32_t)__ldg(sp + 8 + t4) << 16);
                        dd[rt][hl] = h2f(ldg16(base + L.plane[0] + blk * 2));
                        dm[rt][hl] = h2f(ldg16(base + L.plane[1] + blk * 2));
                    }
                }
            }
        }
        // ---- activation fragments of this superblock
        uint4 X[NT], X1[NT];
        float D[NT][2][kTiles][4];
#pragma unroll
        for (int tk = 0; tk < NT; ++tk) {
            const __half* qv = vs.q + (size_t)vec[tk] * vs.q_stride + (size_t)s * 256 + (g * 4 + t4) * 8;
            X[tk] = ldg128(qv + kFam * fam_stride);
            if (FMT == kQ3K) X1[tk] = ldg128(qv + kF1 * fam_stride);
#pragma unroll
            for (int rt = 0; rt < 2; ++rt)
#pragma unroll
                for (int u = 0; u < kTiles; ++u)
#pragma unroll
                    for (int c = 0; c < 4; ++c) D[tk][rt][u][c] = 0.0f;
        }

#pragma unroll
        for (int i = 0; i < 16; ++i) {
            const int owner = kWide ? (i >> 1) : (i & 7);
            const int sel = kWide ? (i & 1) : (i >> 3);
            const int tile = kWide ? 0 : (i >> 3);
            uint32_t q8w[2][2];
            if (FMT == kQ80) {
                // this k-step's 32-bit code word of block i/2 for the 4 rows
#pragma unroll
                for (int rt = 0; rt < 2; ++rt)
#pragma unroll
                    for (int hl = 0; hl < 2; ++hl) {
                        const int b = 8 * s + (i >> 1);
                        q8w[rt][hl] = 0u;
                        if (b < L.blocks_per_row)
                            q8w[rt][hl] = ldg32(base + L.plane[1] + (rowblk[rt][hl] + b) * 32 + 8 * t4 + 4 * (i & 1));
                    }
            }
#pragma unroll
            for (int rt = 0; rt < 2; ++rt) {
                uint32_t a[4], ah[4];
                if (FMT == kQ2K || FMT == kQ3K) {
#pragma unroll
                    for (int hl = 0; hl < 2; ++hl) {
                        const uint32_t w = cw[rt][hl][i >> 2], w10 = w >> 10;
                        switch (i & 3) {
                        case 0: a[hl] = ext2<0>(w, w10); a[2 + hl] = ext2<1>(w, w10); break;
                        case 1: a[hl] = ext2<2>(w, w10); a[2 + hl] = ext2<3>(w, w10); break;
                        case 2: a[hl] = ext2<4>(w, w10); a[2 + hl] = ext2<5>(w, w10); break;
                        default: a[hl] = ext2<6>(w, w10); a[2 + hl] = ext2<7>(w, w10); break;
                        }
                    }
                    if (FMT == kQ3K) {
#pragma unroll
                        for (int hl = 0; hl < 2; ++hl) {
                            const uint32_t w = hw[rt][hl][i >> 3], w10 = w >> 10;
                            switch (i & 7) {
                            case 0: ah[hl] = ext1<0>(w, w10); ah[2 + hl] = ext1<1>(w, w10); break;
                            case 1: ah[hl] = ext1<2>(w, w10); ah[2 + hl] = ext1<3>(w, w10); break;
                            case 2: ah[hl] = ext1<4>(w, w10); ah[2 + hl] = ext1<5>(w, w10); break;
                            case 3: ah[hl] = ext1<6>(w, w10); ah[2 + hl] = ext1<7>(w, w10); break;
                            case 4: ah[hl] = ext1<8>(w, w10); ah[2 + hl] = ext1<9>(w, w10); break;
                            case 5: ah[hl] = ext1<10>(w, w10); ah[2 + hl] = ext1<11>(w, w10); break;
                            case 6: ah[hl] = ext1<12>(w, w10); ah[2 + hl] = ext1<13>(w, w10); break;
                            default: ah[hl] = ext1<14>(w, w10); ah[2 + hl] = ext1<15>(w, w10); break;
                            }
                        }
                    }
                } else if (FMT == kQ4K) {
#pragma unroll
                    for (int hl = 0; hl < 2; ++hl) {
                        const uint32_t w = cw[rt][hl][i >> 1];
                        const uint32_t ws = (i & 1) ? (w >> 8) : w;
                        a[hl] = lop3_and_or(ws, 0x000F000Fu, 0x64006400u);
                        a[2 + hl] = lop3_and_or(ws, 0x00F000F0u, 0x64006400u);
                    }
                } else {  // Q8_0
#pragma unroll
                    for (int hl = 0; hl < 2; ++hl) {
                        a[hl] = lop3_q8(q8w[rt][hl]);
                        a[2 + hl] = lop3_q8(q8w[rt][hl] >> 8);
                    }
                }
#pragma unroll
                for (int tk = 0; tk < NT; ++tk) {
                    const uint32_t b0 = hmul2u(sel ? X[tk].z : X[tk].x, mask[owner]);
                    const uint32_t b1 = hmul2u(sel ? X[tk].w : X[tk].y, mask[owner]);
                    mma16816(D[tk][rt][tile], a[0], a[1], a[2], a[3], b0, b1);
                    if (FMT == kQ3K) {
                        const uint32_t c0 = hmul2u(sel ? X1[tk].z : X1[tk].x, mask[owner]);
                        const uint32_t c1 = hmul2u(sel ? X1[tk].w : X1[tk].y, mask[owner]);
                        mma16816(D[tk][rt][tile], ah[0], ah[1], ah[2], ah[3], c0, c1);
                    }
                }
            }
        }

        // ---- epilogue: sub-block scales / mins, fp32
#pragma unroll
        for (int tk = 0; tk < NT; ++tk) {
            const float* st = vs.st + (size_t)vec[tk] * vs.st_stride;
            if (FMT == kQ2K || FMT == kQ3K) {
                const float4 O = *reinterpret_cast<const float4*>(st + (FMT == kQ2K ? so.os2 : so.oq3) + s * 16 + t4 * 4);
                float4 S = make_float4(0, 0, 0, 0);
                if (FMT == kQ2K) S = *reinterpret_cast<const float4*>(st + so.sxs16 + s * 16 + t4 * 4);
                const float sg0 = st[so.sig + 8 * s + t4], sg1 = st[so.sig + 8 * s + 4 + t4];
                const float Ov[4] = {O.x, O.y, O.z, O.w}, Sv[4] = {S.x, S.y, S.z, S.w};
#pragma unroll
                for (int rt = 0; rt < 2; ++rt) {
#pragma unroll
                    for (int hl = 0; hl < 2; ++hl) {
                        float a_sc = 0.0f, a_m = 0.0f;
#pragma unroll
                        for (int v = 0; v < 4; ++v) {   // v = 2*tile + e
                            const float P = fmaf(D[tk][rt][v >> 1][2 * hl + (v & 1)], (v >> 1) ? sg1 : sg0, -Ov[v]);
                            if (FMT == kQ2K) {
                                const uint32_t byte = (fld[rt][hl] >> (8 * v)) & 0xffu;
                                a_sc = fmaf((float)(byte & 15u), P, a_sc);
                                a_m = fmaf((float)(byte >> 4), Sv[v], a_m);
                            } else {
                                const uint32_t f = fld[rt][hl];
                                const int sfield = (int)((f >> (4 * v)) & 15u) | (int)(((f >> (16 + 2 * v)) & 3u) << 4);
                                a_sc = fmaf((float)(sfield - 32), P, a_sc);
                            }
                        }
                        float r = dd[rt][hl] * a_sc;
                        if (FMT == kQ2K) r = fmaf(-dm[rt][hl], a_m, r);
                        acc[tk][rt][hl] += r;
                    }
                }
            } else {
                const float2 O = *reinterpret_cast<const float2*>(st + (FMT == kQ4K ? so.os4 : so.os8) + 8 * s + 2 * t4);
                const float2 sg = *reinterpret_cast<const float2*>(st + so.sig + 8 * s + 2 * t4);
                float2 S = make_float2(0, 0);
                if (FMT == kQ4K) S = *reinterpret_cast<const float2*>(st + so.sxs32 + 8 * s + 2 * t4);
#pragma unroll
                for (int rt = 0; rt < 2; ++rt) {
#pragma unroll
                    for (int hl = 0; hl < 2; ++hl) {
                        const float P0 = fmaf(D[tk][rt][0][2 * hl], sg.x, -O.x);
                        const float P1 = fmaf(D[tk][rt][0][2 * hl + 1], sg.y, -O.y);
                        if (FMT == kQ4K) {
                            const uint32_t f = fld[rt][hl];
                            const int hi = (int)(f >> 16);
                            const float sc0 = (float)((f & 15u) | ((hi & 3) << 4));
                            const float m0 = (float)(((f >> 4) & 15u) | (((hi >> 2) & 3) << 4));
                            const float sc1 = (float)(((f >> 8) & 15u) | (((hi >> 4) & 3) << 4));
                            const float m1 = (float)(((f >> 12) & 15u) | (((hi >> 6) & 3) << 4));
                            const float a_sc = fmaf(sc1, P1, sc0 * P0);
                            const float a_m = fmaf(m1, S.y, m0 * S.x);
                            acc[tk][rt][hl] += fmaf(dd[rt][hl], a_sc, -dm[rt][hl] * a_m);
                        } else {
                            acc[tk][rt][hl] += fmaf(dd[rt][hl], P0, dm[rt][hl] * P1);
                        }
                    }
                }
            }
        }
    }
}

struct DecodeArgs {
    Dims d;
    int nsbx, nsbi;          // superblocks along hidden / inter
    const __half* xq; const float* xs;   // prepared tokens
    __half* hq; float* hs;               // prepared SwiGLU outputs (per assignment)
    const int32_t* offsets; const int32_t* perm; const int32_t* active; const float* wts;
    float* pgu;              // [A][2][kMaxSplit][I]
    float* pdn;              // [A][H]
    uint32_t* gu_cnt;        // [(E+1) * I/32]
    uint32_t* dn_cnt;        // [H/32]
    uint32_t* next;          // [2] item counters
    float* out;
};

__device__ __forceinline__ int nsplit_gu(int fmt) { return fmt == kQ80 ? 4 : fmt == kQ4K ? 2 : 1; }

// tokens of expert slot: returns count; tok(q) gives (vector id for x, assignment id)
struct SlotTokens {
    int e, first, n;
    bool shared;
};
__device__ __forceinline__ SlotTokens slot_tokens(const DecodeArgs& A, int slotpos) {
    SlotTokens st;
    if (slotpos < A.d.has_shared) { st.shared = true; st.e = A.d.E; st.first = 0; st.n = A.d.T; }
    else {
        st.shared = false;
        st.e = A.active[1 + slotpos - A.d.has_shared];
        st.first = A.offsets[st.e];
        st.n = A.offsets[st.e + 1] - st.first;
    }
    return st;
}
__device__ __forceinline__ void token_of(const DecodeArgs& A, const SlotTokens& st, int q, int& t, int& a) {
    if (st.shared) { t = q; a = A.d.T * A.d.K + q; }
    else { a = A.perm[st.first + q]; t = a / A.d.K; }
}

template <int NT>
__device__ __forceinline__ void run_gemv(int fmt, const uint8_t* base, const TensorLayout& L, int row0, int sb0,
                                         int sb1, const int (&vec)[NT], const VecSrc& vs, float (&acc)[NT][2][2]) {
    switch (fmt) {
    case kQ2K: gemv_item<kQ2K, NT>(base, L, row0, sb0, sb1, vec, vs, acc); break;
    case kQ3K: gemv_item<kQ3K, NT>(base, L, row0, sb0, sb1, vec, vs, acc); break;
    case kQ4K: gemv_item<kQ4K, NT>(base, L, row0, sb0, sb1, vec, vs, acc); break;
    default: gemv_item<kQ80, NT>(base, L, row0, sb0, sb1, vec, vs, acc); break;
    }
}

// reduce acc over the 4 lanes sharing g; lanes with t4 == 0 store rows
template <int NT>
__device__ __forceinline__ void store_rows(const float (&acc)[NT][2][2], int ntok, float* const (&dst)[NT], int row0) {
    const int lane = threadIdx.x & 31, g = lane >> 2, t4 = lane & 3;
#pragma unroll
    for (int tk = 0; tk < NT; ++tk) {
#pragma unroll
        for (int rt = 0; rt < 2; ++rt)
#pragma unroll
            for (int hl = 0; hl < 2; ++hl) {
                float v = acc[tk][rt][hl];
                v += __shfl_xor_sync(kFull, v, 1);
                v += __shfl_xor_sync(kFull, v, 2);
                if (t4 == 0 && tk < ntok) dst[tk][row0 + 16 * rt + 8 * hl + g] = v;
            }
    }
}

__global__ void __launch_bounds__(kWarpsPerCta * 32, 2) gateup_mma_kernel(const __grid_constant__ ExpertTab tab,
                                                                          const __grid_constant__ DecodeArgs A) {
    const int lane = threadIdx.x & 31;
    const Dims& d = A.d;
    const int n_rb = d.I / 32;
    const int n_slots = A.active[0] + d.has_shared;
    const int total = n_slots * 2 * n_rb * kMaxSplit;
    const int n_assign = d.T * d.K + d.T;
    const VecSrc vs{A.xq, A.xs, (size_t)4 * A.nsbx * 256, (size_t)stat_off(A.nsbx).total, A.nsbx};
    for (;;) {
        int item = 0;
        if (lane == 0) item = (int)atomicAdd(&A.next[0], 1u);
        item = __shfl_sync(kFull, item, 0);
        if (item >= total) break;
        const int ks = item % kMaxSplit;
        int rest = item / kMaxSplit;
        const int rb = rest % n_rb;
        rest /= n_rb;
        const int tensor = rest & 1, slotpos = rest >> 1;
        const SlotTokens stk = slot_tokens(A, slotpos);
        const int fmt = tab.fmt[stk.e][tensor];
        const int ns = nsplit_gu(fmt);
        if (ks >= ns) continue;
        const int sb0 = ks * A.nsbx / ns, sb1 = (ks + 1) * A.nsbx / ns;
        const TensorLayout L = tensor_layout(fmt, d.I, d.H);
        const uint8_t* base = tab.p[stk.e][tensor];
        for (int q0 = 0; q0 < stk.n; q0 += 2) {
            if (stk.n - q0 == 1) {
                int t, a; token_of(A, stk, q0, t, a);
                int vec[1] = {t};
                float acc[1][2][2] = {};
                run_gemv<1>(fmt, base, L, 32 * rb, sb0, sb1, vec, vs, acc);
                float* dst[1] = {A.pgu + ((size_t)a * 2 * kMaxSplit + tensor * kMaxSplit + ks) * d.I};
                store_rows<1>(acc, 1, dst, 32 * rb);
            } else {
                int t0, a0, t1, a1;
                token_of(A, stk, q0, t0, a0);
                token_of(A, stk, q0 + 1, t1, a1);
                int vec[2] = {t0, t1};
                float acc[2][2][2] = {};
                run_gemv<2>(fmt, base, L, 32 * rb, sb0, sb1, vec, vs, acc);
                float* dst[2] = {A.pgu + ((size_t)a0 * 2 * kMaxSplit + tensor * kMaxSplit + ks) * d.I,
                                 A.pgu + ((size_t)a1 * 2 * kMaxSplit + tensor * kMaxSplit + ks) * d.I};
                store_rows<2>(acc, 2, dst, 32 * rb);
            }
        }
        // last warp of this (expert, row block): SwiGLU + prepare h for the down projection
        __threadfence();
        __syncwarp();
        const int target = nsplit_gu(tab.fmt[stk.e][0]) + nsplit_gu(tab.fmt[stk.e][1]);
        unsigned prev = 0;
        if (lane == 0) prev = atomicAdd(&A.gu_cnt[slotpos * n_rb + rb], 1u);
        prev = __shfl_sync(kFull, prev, 0);
        if ((int)prev + 1 != target) continue;
        __threadfence();
        const int ngs = nsplit_gu(tab.fmt[stk.e][0]), nus = nsplit_gu(tab.fmt[stk.e][1]);
        const int fam = families_of(tab.fmt[stk.e][2]);
        const int row = 32 * rb + lane;
        for (int q = 0; q < stk.n; ++q) {
            int t, a; token_of(A, stk, q, t, a);
            const float* pg = A.pgu + (size_t)a * 2 * kMaxSplit * d.I;
            float gs = 0.0f, us = 0.0f;
            for (int k = 0; k < ngs; ++k) gs += __ldcg(pg + (size_t)k * d.I + row);
            for (int k = 0; k < nus; ++k) us += __ldcg(pg + (size_t)(kMaxSplit + k) * d.I + row);
            const float w = stk.shared ? 1.0f : A.wts[a];
            const float h = gs / (1.0f + expf(-gs)) * us * w;
            __half* hq = A.hq + (size_t)a * 4 * A.nsbi * 256;
            float* hs = A.hs + (size_t)a * stat_off(A.nsbi).total;
            prep_block32(h, rb, fam, hq, hs, A.nsbi);
            // the warp that finishes the last row block also zero-fills the
            // padding of the last superblock (inter not a multiple of 256)
            if (rb == n_rb - 1)
                for (int jb = n_rb; jb < 8 * A.nsbi; ++jb) prep_block32(0.0f, jb, fam, hq, hs, A.nsbi);
        }
        (void)n_assign;
    }
}

__global__ void __launch_bounds__(kWarpsPerCta * 32, 2) down_mma_kernel(const __grid_constant__ ExpertTab tab,
                                                                        const __grid_constant__ DecodeArgs A) {
    const int lane = threadIdx.x & 31;
    const Dims& d = A.d;
    const int n_rb = d.H / 32;
    const int n_slots = A.active[0] + d.has_shared;
    const int total = n_slots * n_rb;
    const VecSrc vs{A.hq, A.hs, (size_t)4 * A.nsbi * 256, (size_t)stat_off(A.nsbi).total, A.nsbi};
    for (;;) {
        int item = 0;
        if (lane == 0) item = (int)atomicAdd(&A.next[1], 1u);
        item = __shfl_sync(kFull, item, 0);
        if (item >= total) break;
        const int slotpos = item / n_rb, rb = item % n_rb;
        const SlotTokens stk = slot_tokens(A, slotpos);
        const int fmt = tab.fmt[stk.e][2];
        const TensorLayout L = tensor_layout(fmt, d.H, d.I);
        const uint8_t* base = tab.p[stk.e][2];
        for (int q0 = 0; q0 < stk.n; q0 += 2) {
            if (stk.n - q0 == 1) {
                int t, a; token_of(A, stk, q0, t, a);
                int vec[1] = {a};
                float acc[1][2][2] = {};
                run_gemv<1>(fmt, base, L, 32 * rb, 0, A.nsbi, vec, vs, acc);
                float* dst[1] = {A.pdn + (size_t)a * d.H};
                store_rows<1>(acc, 1, dst, 32 * rb);
            } else {
                int t0, a0, t1, a1;
                token_of(A, stk, q0, t0, a0);
                token_of(A, stk, q0 + 1, t1, a1);
                int vec[2] = {a0, a1};
                float acc[2][2][2] = {};
                run_gemv<2>(fmt, base, L, 32 * rb, 0, A.nsbi, vec, vs, acc);
                float* dst[2] = {A.pdn + (size_t)a0 * d.H, A.pdn + (size_t)a1 * d.H};
                store_rows<2>(acc, 2, dst, 32 * rb);
            }
        }
        __threadfence();
        __syncwarp();
        unsigned prev = 0;
        if (lane == 0) prev = atomicAdd(&A.dn_cnt[rb], 1u);
        prev = __shfl_sync(kFull, prev, 0);
        if ((int)prev + 1 != n_slots) continue;
        __threadfence();
        // combine: routed experts in slot order (weights already folded into h), then shared
        const int row = 32 * rb + lane;
        for (int t = 0; t < d.T; ++t) {
            float y = 0.0f;
            for (int j = 0; j < d.K; ++j) y += __ldcg(A.pdn + (size_t)(t * d.K + j) * d.H + row);
            if (d.has_shared) y += __ldcg(A.pdn + (size_t)(d.T * d.K + t) * d.H + row);
            A.out[(size_t)t * d.H + row] = y;
        }
    }
}

int g_num_sms = 0;

}  // namespace

size_t decode_scratch_bytes(const Dims& d) {
    const size_t A = (size_t)d.T * d.K + d.T;
    const int nsbi = (d.I + 255) / 256;
    size_t b = 0;
    b += A * 4 * nsbi * 256 * 2;                 // hq
    b += A * stat_off(nsbi).total * 4;           // hs
    b += A * 2 * kMaxSplit * d.I * 4;            // pgu
    b += A * d.H * 4;                            // pdn
    return b + 4 * 256;
}

size_t decode_counter_bytes(const Dims& d) {
    return ((size_t)(d.E + 1) * (d.I / 32) + d.H / 32 + 2) * 4;
}

cudaError_t launch_decode_mma(const Dims& d, const ExpertTab& tab, const Work& w, float* out, cudaStream_t s) {
    if (d.T == 0) return cudaSuccess;
    if (g_num_sms == 0) {
        int dev = 0;
        cudaGetDevice(&dev);
        cudaDeviceGetAttribute(&g_num_sms, cudaDevAttrMultiProcessorCount, dev);
        if (g_num_sms <= 0) g_num_sms = 148;
    }
    DecodeArgs A;
    A.d = d;
    A.nsbx = (d.H + 255) / 256;
    A.nsbi = (d.I + 255) / 256;
    A.xq = w.xq; A.xs = w.xs; A.hq = w.hq; A.hs = w.hs;
    A.offsets = w.offsets; A.perm = w.perm; A.active = w.active; A.wts = w.wts;
    A.pgu = w.pgu; A.pdn = w.pdn;
    A.gu_cnt = w.counters; A.dn_cnt = w.counters + (size_t)(d.E + 1) * (d.I / 32);
    A.next = A.dn_cnt + d.H / 32;
    A.out = out;
    const int grid = g_num_sms * 2;
    prof_begin("gateup_mma", s);
    gateup_mma_kernel<<<grid, kWarpsPerCta * 32, 0, s>>>(tab, A);
    prof_end(s);
    cudaError_t err = cudaGetLastError();
    if (err != cudaSuccess) return err;
    prof_begin("down_mma", s);
    down_mma_kernel<<<grid, kWarpsPerCta * 32, 0, s>>>(tab, A);
    prof_end(s);
    return cudaGetLastError();
}

}  // namespace mq
