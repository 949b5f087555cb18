// Expert FFN for decode-sized batches on the tcgen05 tensor cores
// (arXiv 2509.25689 Fig. 1: a shared expert plus router-weighted routed
// SwiGLU experts; each expert tensor in its own k-quant style format, Sec. 3.3).
//
// A CTA holds two groups of 4 warps; a group owns 128 weight rows (thread =
// row = tensor-memory lane).  The contraction runs in units of 128 positions
// (half a superblock).  Per unit every thread
//   * turns its row's packed codes into fp16 MMA operands with one AND per
//     code pair (the code lands in the mantissa of an fp16 subnormal, value
//     code * 2^(s-24); the prepared activation carries 2^-s) and stores them
//     to tensor memory (tcgen05.st): A = 128 rows x 128 positions;
//   * the first 16 x (tokens) threads copy 8 prepared activations each into
//     the unit's B matrices in shared memory: K-step q (16 positions) has one
//     nonzero column per token, the column of the sub-block q belongs to, so
//     D = A B holds per-(row, sub-block, token) sums;
// and one thread issues the unit's 8 MMAs (M 128, N 16 or 32, K 16, fp32 in
// tensor memory).  The MMAs run while the threads read back the previous
// unit's D (tcgen05.ld) and apply its sub-block scales and mins in fp32.
// Weights come straight from global memory into registers, 4 units ahead.
// Gate/up CTAs run the gate rows in one group and the same up rows in the
// other and finish with SwiGLU (routing weight folded in) and the prepared h
// of the down projection; down CTAs run one 128-row item per group and write
// one partial output row block per assignment.  Every wait on an mbarrier is
// bounded (about 1 s) and reports to the error word; a failure stops the
// group (gate/up: the CTA) at the next item boundary; tensor memory is freed
// on every exit path.
#include <cuda_fp16.h>

#include "mq_actprep.cuh"
#include "mq_internal.h"

namespace mq {
namespace {

constexpr int kTThreads = 256;               // two groups of 4 warps
constexpr int kRowsT = 128;                  // weight rows per group (MMA M)
constexpr int kNB = 32;                      // B matrix rows (token x sub-block columns)
constexpr int kBMat = kNB * 16 * 2;          // bytes of one B matrix (1 KB)
constexpr int kBBuf = 8 * kBMat;             // one unit's 8 matrices
constexpr uint32_t kErrT = 8u;
constexpr int kMaxCachedAssign = 1024;

__device__ __forceinline__ uint64_t global_ns() {
    uint64_t t;
    asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
    return t;
}
__device__ __forceinline__ bool mbar_try(uint32_t bar, uint32_t parity) {
    uint32_t ok;
    asm volatile(
        "{\n\t.reg .pred p;\n\tmbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\tselp.u32 %0, 1, 0, p;\n\t}"
        : "=r"(ok) : "r"(bar), "r"(parity) : "memory");
    return ok != 0;
}
// Bounded wait (about 1 s).  Once a wait of this thread has given up, later
// ones return at once, so a broken pipeline costs one timeout per thread.
__device__ __forceinline__ void mbar_wait(uint32_t bar, uint32_t parity, bool& alive) {
    if (!alive || mbar_try(bar, parity)) return;
    const uint64_t t0 = global_ns();
    for (;;) {
        if (mbar_try(bar, parity)) return;
        if (global_ns() - t0 > 1000000000ull) { alive = false; return; }
    }
}
__device__ __forceinline__ uint64_t sdesc(uint32_t saddr, uint32_t lbo, uint32_t sbo) {
    return (uint64_t)((saddr & 0x3FFFFu) >> 4) | ((uint64_t)((lbo >> 4) & 0x3FFFu) << 16) |
           ((uint64_t)((sbo >> 4) & 0x3FFFu) << 32) | ((uint64_t)1 << 46);
}
// kind::f16 instruction descriptor: fp32 accumulator, fp16 A and B, both K-major
__device__ __forceinline__ uint32_t idesc_f16(int M, int N) {
    return (1u << 4) | ((uint32_t)(N >> 3) << 17) | ((uint32_t)(M >> 4) << 24);
}
__device__ __forceinline__ uint4 ldg128(const void* p) { return __ldg(reinterpret_cast<const uint4*>(p)); }
__device__ __forceinline__ uint32_t ldg32(const void* p) { return __ldg(reinterpret_cast<const unsigned int*>(p)); }
__device__ __forceinline__ uint32_t ldg16(const void* p) { return __ldg(reinterpret_cast<const unsigned short*>(p)); }
__device__ __forceinline__ float h2f(uint32_t bits16) {
    return __half2float(__ushort_as_half((unsigned short)(bits16 & 0xffffu)));
}
__device__ __forceinline__ uint32_t sub4(const uint4& v, int i) {
    return i == 0 ? v.x : i == 1 ? v.y : i == 2 ? v.z : v.w;
}
__device__ __forceinline__ void group_sync(int grp) {
    asm volatile("bar.sync %0, %1;" ::"r"(1 + grp), "n"(128) : "memory");
}
// barrier over the group that also ORs a predicate across it
__device__ __forceinline__ bool group_any(int grp, bool v) {
    uint32_t r;
    asm volatile("{\n\t.reg .pred p, q;\n\tsetp.ne.u32 p, %1, 0;\n\tbar.red.or.pred q, %2, %3, p;\n\t"
                 "selp.u32 %0, 1, 0, q;\n\t}"
                 : "=r"(r) : "r"((uint32_t)v), "r"(1 + grp), "n"(128) : "memory");
    return r != 0;
}
__device__ __forceinline__ void tmem_st32(uint32_t taddr, const uint32_t (&r)[32]) {
    asm volatile(
        "tcgen05.st.sync.aligned.32x32b.x32.b32 [%0], {%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,%16,"
        "%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31,%32};"
        ::"r"(taddr), "r"(r[0]), "r"(r[1]), "r"(r[2]), "r"(r[3]), "r"(r[4]), "r"(r[5]), "r"(r[6]), "r"(r[7]),
          "r"(r[8]), "r"(r[9]), "r"(r[10]), "r"(r[11]), "r"(r[12]), "r"(r[13]), "r"(r[14]), "r"(r[15]),
          "r"(r[16]), "r"(r[17]), "r"(r[18]), "r"(r[19]), "r"(r[20]), "r"(r[21]), "r"(r[22]), "r"(r[23]),
          "r"(r[24]), "r"(r[25]), "r"(r[26]), "r"(r[27]), "r"(r[28]), "r"(r[29]), "r"(r[30]), "r"(r[31])
        : "memory");
}
__device__ __forceinline__ void tmem_ld8(uint32_t taddr, uint32_t (&r)[8]) {
    asm volatile("tcgen05.ld.sync.aligned.32x32b.x8.b32 {%0,%1,%2,%3,%4,%5,%6,%7}, [%8];"
                 : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7])
                 : "r"(taddr)
                 : "memory");
}
__device__ __forceinline__ void tmem_ld4(uint32_t taddr, uint32_t (&r)[8]) {
    asm volatile("tcgen05.ld.sync.aligned.32x32b.x4.b32 {%0,%1,%2,%3}, [%4];"
                 : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3])
                 : "r"(taddr)
                 : "memory");
}

struct TArgs {
    Dims d;
    int nsbx, nsbi;
    const __half* xq; const float* xs;   // prepared tokens
    __half* hq; float* hs;               // prepared SwiGLU outputs (per assignment)
    const int32_t* offsets; const int32_t* perm; const int32_t* active; const float* wts;
    float* pdn;
    uint32_t* err;
};

struct TSlots {
    int32_t first[kMaxExperts + 1], ntot[kMaxExperts + 1], pre[kMaxExperts + 2];
    const uint8_t* ptr[kMaxExperts + 1][2];
    uint8_t fmt[kMaxExperts + 1][2];
    uint8_t down_fmt[kMaxExperts + 1];
};

// ---- packed fields of one row ----------------------------------------------
// Sc: what the epilogue of one unit needs; Raw: one load step (Q2_K / Q3_K:
// a superblock = 2 units, read with 16-byte loads; Q4_K / Q8_0: one unit).
template <int FMT> struct Sc;
template <> struct Sc<kQ2K> { uint4 f; uint32_t dd; };        // 16 scale|min bytes (slot order), d | dmin
template <> struct Sc<kQ3K> { uint32_t s[3]; uint32_t d; };   // 12 scale bytes, d
template <> struct Sc<kQ4K> { uint32_t s[3]; uint32_t dd; };  // 12 scale bytes, d | dmin
template <> struct Sc<kQ80> { uint32_t d[4]; };               // d of the unit's 4 blocks
template <int FMT> struct Raw;
template <> struct Raw<kQ2K> { uint4 c[4]; Sc<kQ2K> sc; };
template <> struct Raw<kQ3K> { uint4 c[4]; uint4 h[2]; Sc<kQ3K> sc; };
template <> struct Raw<kQ4K> { uint4 c[4]; Sc<kQ4K> sc; };
template <> struct Raw<kQ80> { uint4 c[8]; Sc<kQ80> sc; };

template <int FMT> struct TCfg {
    static constexpr int G = (FMT == kQ2K || FMT == kQ3K) ? 2 : 1;   // units per load step
    static constexpr int NB = FMT == kQ4K ? 4 : 2;                     // load steps in flight
};

// Plane pointers of one row: the record of superblock (Q8_0: block) b of
// plane p is at row[p] + b * step[p] (rows are tiled by 32).
struct RowP { const uint8_t* row[4]; int step[4]; int nblk; };
__device__ __forceinline__ RowP row_planes(int fmt, const uint8_t* base, int64_t rows, int64_t cols, int64_t R) {
    const TensorLayout L = tensor_layout(fmt, rows, cols);
    const PlaneBytes pb = plane_bytes(fmt);
    RowP P;
    P.nblk = (int)L.blocks_per_row;
#pragma unroll
    for (int p = 0; p < 4; ++p) {
        P.row[p] = p < pb.n ? rec_ptr(base + L.plane[p], L, pb.b[p], R, 0) : base;
        P.step[p] = p < pb.n ? kRowTile * pb.b[p] : 0;
    }
    return P;
}

template <int FMT>
__device__ __forceinline__ void load_step(const RowP& P, int s, Raw<FMT>& R) {
    if constexpr (FMT == kQ2K) {
        const uint8_t* c = P.row[3] + (size_t)s * P.step[3];
#pragma unroll
        for (int i = 0; i < 4; ++i) R.c[i] = ldg128(c + 16 * i);
        R.sc.f = ldg128(P.row[2] + (size_t)s * P.step[2]);
        R.sc.dd = ldg16(P.row[0] + (size_t)s * P.step[0]) | (ldg16(P.row[1] + (size_t)s * P.step[1]) << 16);
    } else if constexpr (FMT == kQ3K) {
        const uint8_t* c = P.row[2] + (size_t)s * P.step[2];
#pragma unroll
        for (int i = 0; i < 4; ++i) R.c[i] = ldg128(c + 16 * i);
        const uint8_t* h = P.row[3] + (size_t)s * P.step[3];
        R.h[0] = ldg128(h);
        R.h[1] = ldg128(h + 16);
        const uint8_t* f = P.row[1] + (size_t)s * P.step[1];
        R.sc.s[0] = ldg32(f); R.sc.s[1] = ldg32(f + 4); R.sc.s[2] = ldg32(f + 8);
        R.sc.d = ldg16(P.row[0] + (size_t)s * P.step[0]);
    } else if constexpr (FMT == kQ4K) {
        // unit s = half s & 1 of superblock s >> 1: the record's 64-byte unit s & 1
        const int sb = s >> 1;
        const uint8_t* c = P.row[3] + (size_t)sb * P.step[3] + (s & 1) * (kRowTile * 64);
#pragma unroll
        for (int i = 0; i < 4; ++i) R.c[i] = ldg128(c + 16 * i);
        const uint8_t* f = P.row[2] + (size_t)sb * P.step[2];
        R.sc.s[0] = ldg32(f); R.sc.s[1] = ldg32(f + 4); R.sc.s[2] = ldg32(f + 8);
        R.sc.dd = ldg16(P.row[0] + (size_t)sb * P.step[0]) | (ldg16(P.row[1] + (size_t)sb * P.step[1]) << 16);
    } else {
#pragma unroll
        for (int i = 0; i < 4; ++i) {
            // blocks past the row's last one (columns padded to 256) read as
            // zero; their activations are zero too
            const int b = 4 * s + i;
            R.c[2 * i] = R.c[2 * i + 1] = make_uint4(0u, 0u, 0u, 0u);
            R.sc.d[i] = 0u;
            if (b < P.nblk) {
                const uint8_t* c = P.row[1] + (size_t)b * P.step[1];
                R.c[2 * i] = ldg128(c);
                R.c[2 * i + 1] = ldg128(c + 16);
                R.sc.d[i] = ldg16(P.row[0] + (size_t)b * P.step[0]);
            }
        }
    }
}

// The unit's A operand: 64 columns of fp16 pairs (K-step q = columns 8q ..
// 8q + 7, pair m in column 8q + m), written to tensor memory at taddr.
// hh: which half of the superblock (Q2_K / Q3_K raw steps hold both).
template <int FMT>
__device__ __forceinline__ void store_a(const Raw<FMT>& R, int hh, uint32_t taddr) {
#pragma unroll
    for (int half = 0; half < 2; ++half) {
        uint32_t a[32];
#pragma unroll
        for (int qq = 0; qq < 4; ++qq) {
            const int q = 4 * half + qq;
#pragma unroll
            for (int m = 0; m < 8; ++m) {
                uint32_t v;
                if constexpr (FMT == kQ2K) {
                    // sub-block j = 8 hh + q in word 4 (q & 3) + 2 hh + (q >> 2), pair m at bit 2m
                    const uint32_t w = sub4(R.c[q & 3], 2 * hh + (q >> 2));
                    v = m <= 4 ? (w & (0x00030003u << (2 * m))) : ((w >> 10) & (0x00030003u << (2 * (m - 5))));
                } else if constexpr (FMT == kQ3K) {
                    // low bits as Q2_K; high bit in word 2 (q & 3) + hh at bit 8 (q >> 2) + m:
                    // the full 3-bit code, unscaled
                    const uint32_t wl = sub4(R.c[q & 3], 2 * hh + (q >> 2));
                    const int wi = 2 * (q & 3) + hh;
                    const uint32_t wh = sub4(R.h[wi >> 2], wi & 3) >> (8 * (q >> 2));
                    v = ((wl >> (2 * m)) & 0x00030003u) | (((wh >> m) & 0x00010001u) << 2);
                } else if constexpr (FMT == kQ4K) {
                    // sub-block q >> 1 of the unit, pair p = 8 (q & 1) + m: word 4 (q >> 1) + p / 4, bit 4 (p % 4)
                    const int p = 8 * (q & 1) + m;
                    const uint32_t w = sub4(R.c[q >> 1], p >> 2);
                    v = ((p & 2) ? (w >> 8) : w) & ((p & 1) ? 0x00F000F0u : 0x000F000Fu);
                } else {
                    // block q >> 1 of the unit, pair p = 8 (q & 1) + m: word p / 2 of the block, byte p % 2
                    const int p = 8 * (q & 1) + m;
                    const uint32_t w = sub4(R.c[2 * (q >> 1) + (p >> 3)], (p >> 1) & 3);
                    v = ((p & 1) ? (w >> 8) : w) & 0x00FF00FFu;
                }
                a[8 * qq + m] = v;
            }
        }
        tmem_st32(taddr + 32 * half, a);
    }
}

// Prepared activation family matching each format's A values: Q2_K pairs
// carry 4^m-style positional powers (F2), Q3_K 3-bit codes none (F8), Q4_K
// 16^(m & 1) (F4), Q8_0 none (F8).
__host__ __device__ __forceinline__ int tfam(int fmt) { return fmt == kQ2K ? kF2 : fmt == kQ4K ? kF4 : kF8; }
// B column (= D column) of token tk for K-step q of a unit
template <int FMT>
__device__ __forceinline__ int bcol(int tk, int q) {
    return (FMT == kQ2K || FMT == kQ3K) ? 8 * tk + q : 4 * tk + (q >> 1);
}

// Epilogue of unit u for this thread's row: reads the unit's D columns of
// each token from tensor memory (taddr: the D buffer, this warp's lanes) and
// applies the sub-block scales and mins.
template <int FMT>
__device__ __forceinline__ void epilogue(const Sc<FMT>& S, int u, uint32_t taddr, int ntok,
                                         const float* const (&st)[kDecodeTok], float (&acc)[kDecodeTok]) {
    const int s = u >> 1, hh = u & 1;
#pragma unroll
    for (int tk = 0; tk < kDecodeTok; ++tk) {
        if (tk >= ntok) break;
        uint32_t dv[8];
        if constexpr (FMT == kQ2K || FMT == kQ3K) tmem_ld8(taddr + 8 * tk, dv);
        else tmem_ld4(taddr + 4 * tk, dv);
        const float* rec = st[tk] + (size_t)s * kStatFloats;
        const float4 cf = __ldg(reinterpret_cast<const float4*>(rec + kStatC + 4 * hh));
        asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
        if constexpr (FMT == kQ2K) {
            // d * sc * sum(q v) - dmin * m * sum(v) per 16-wide sub-block j = 8 hh + q;
            // the sums of sub-blocks 8 hh + 2t, 8 hh + 2t + 1 sit in slots 4t + 2 hh, 4t + 2 hh + 1
            float a = 0.0f, am = 0.0f;
#pragma unroll
            for (int t = 0; t < 4; ++t) {
                const float2 sv = __ldg(reinterpret_cast<const float2*>(rec + kStatS16 + 4 * t + 2 * hh));
                const float c = t == 0 ? cf.x : t == 1 ? cf.y : t == 2 ? cf.z : cf.w;
                const uint32_t w = sub4(S.f, t) >> (16 * hh);
                a = fmaf((float)(w & 15u) * c, __uint_as_float(dv[2 * t]), a);
                a = fmaf((float)((w >> 8) & 15u) * c, __uint_as_float(dv[2 * t + 1]), a);
                am = fmaf((float)((w >> 4) & 15u), sv.x, am);
                am = fmaf((float)((w >> 12) & 15u), sv.y, am);
            }
            acc[tk] += fmaf(h2f(S.dd), a, -h2f(S.dd >> 16) * am);
        } else if constexpr (FMT == kQ3K) {
            // d * (s - 32) * (sum(c v) - 4 sum(v)), c the 3-bit code
            float a = 0.0f;
#pragma unroll
            for (int t = 0; t < 4; ++t) {
                const float2 sv = __ldg(reinterpret_cast<const float2*>(rec + kStatS16 + 4 * t + 2 * hh));
                const float c = t == 0 ? cf.x : t == 1 ? cf.y : t == 2 ? cf.z : cf.w;
#pragma unroll
                for (int e = 0; e < 2; ++e) {
                    const int u6 = 4 * t + 2 * hh + e;   // slot of sub-block 8 hh + 2t + e
                    const uint32_t lo = (t < 2 ? (S.s[0] >> (8 * (2 * t + hh))) : (S.s[1] >> (8 * (2 * t - 4 + hh))))
                                        >> (4 * e);
                    const uint32_t hi = S.s[2] >> (8 * t + 2 * (2 * hh + e));
                    const float sc = (float)((int)((lo & 15u) | ((hi & 3u) << 4)) - 32);
                    (void)u6;
                    a = fmaf(sc, fmaf(__uint_as_float(dv[2 * t + e]), c, -4.0f * (e ? sv.y : sv.x)), a);
                }
            }
            acc[tk] = fmaf(h2f(S.d), a, acc[tk]);
        } else if constexpr (FMT == kQ4K) {
            // d * sc * sum(q v) - dmin * m * sum(v) per 32-wide sub-block j = 4 hh + jj
            const float4 s32 = __ldg(reinterpret_cast<const float4*>(rec + kStatS32 + 4 * hh));
            const uint32_t lo4 = hh ? S.s[1] : S.s[0];
            const uint32_t hi4 = S.s[2] >> (16 * hh);
            float a = 0.0f, am = 0.0f;
#pragma unroll
            for (int jj = 0; jj < 4; ++jj) {
                const uint32_t lo = lo4 >> (8 * jj), high = hi4 >> (4 * jj);
                const float sc = (float)((lo & 15u) | ((high & 3u) << 4));
                const float mn = (float)(((lo >> 4) & 15u) | (((high >> 2) & 3u) << 4));
                const float c = jj == 0 ? cf.x : jj == 1 ? cf.y : jj == 2 ? cf.z : cf.w;
                const float sm = jj == 0 ? s32.x : jj == 1 ? s32.y : jj == 2 ? s32.z : s32.w;
                a = fmaf(sc * c, __uint_as_float(dv[jj]), a);
                am = fmaf(mn, sm, am);
            }
            acc[tk] += fmaf(h2f(S.dd), a, -h2f(S.dd >> 16) * am);
        } else {
            // d * (sum((q + 128) v) - 128 sum(v)) per block
            const float4 s32 = __ldg(reinterpret_cast<const float4*>(rec + kStatS32 + 4 * hh));
#pragma unroll
            for (int i = 0; i < 4; ++i) {
                const float c = i == 0 ? cf.x : i == 1 ? cf.y : i == 2 ? cf.z : cf.w;
                const float sm = i == 0 ? s32.x : i == 1 ? s32.y : i == 2 ? s32.z : s32.w;
                acc[tk] = fmaf(h2f(S.d[i]), fmaf(__uint_as_float(dv[i]), c, -128.0f * sm), acc[tk]);
            }
        }
    }
}

// Group context of one tensor pass.
struct GCtx {
    uint32_t tA, tD;    // tensor memory: A buffers (2 x 64 columns), D buffers (2 x 32 columns)
    uint32_t bsm;       // shared memory: B buffers (2 x kBBuf)
    uint32_t bar;       // 2 mbarriers (one per buffer)
    uint32_t lane_off;  // this warp's lane quarter
    int grp;
    bool leader;
};

// One tensor of one item for this group: the dot products of 128 rows with
// up to kDecodeTok activation vectors over n_units units.  xsrc: this
// thread's 16-byte slice of the B data (null when it writes none) and boff
// its place in a B buffer; uc: the group's running unit count (buffer and
// mbarrier phase).
template <int FMT>
__device__ __noinline__ void run_tensor(const GCtx& g, const RowP& P, int n_units, int ntok, const __half* xsrc,
                                           int boff, const float* const (&st)[kDecodeTok], int& uc, bool& alive,
                                           float (&acc)[kDecodeTok]) {
    constexpr int G = TCfg<FMT>::G, NB = TCfg<FMT>::NB;
    const int npad = (bcol<FMT>(ntok - 1, 7) + 1 + 15) & ~15;
    const uint32_t idesc = idesc_f16(kRowsT, npad);
    const int n_steps = n_units / G;
    Raw<FMT> R[NB];
    uint4 XB[NB][G];
#pragma unroll
    for (int b = 0; b < NB; ++b) {
        if (b < n_steps) {
            load_step<FMT>(P, b, R[b]);
#pragma unroll
            for (int gg = 0; gg < G; ++gg)
                if (xsrc) XB[b][gg] = ldg128(xsrc + (size_t)128 * (b * G + gg));
        }
    }
    Sc<FMT> prev = R[0].sc;
    for (int k = 0; k < n_steps; k += NB) {
#pragma unroll
        for (int b = 0; b < NB; ++b) {
            const int s = k + b;
            if (s >= n_steps) break;
#pragma unroll
            for (int gg = 0; gg < G; ++gg) {
                const int u = s * G + gg;
                const int buf = uc & 1;
                // (1) operands of unit u
                store_a<FMT>(R[b], G == 2 ? gg : 0, g.tA + buf * 64 + g.lane_off);
                if (xsrc) {
                    const uint4 v = XB[b][gg];
                    asm volatile("st.shared.v4.u32 [%0], {%1,%2,%3,%4};"
                                 ::"r"(g.bsm + buf * kBBuf + boff), "r"(v.x), "r"(v.y), "r"(v.z), "r"(v.w)
                                 : "memory");
                }
                asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory");
                asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
                asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
                group_sync(g.grp);
                if (g.leader) {
                    asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
#pragma unroll
                    for (int q = 0; q < 8; ++q) {
                        const uint64_t db = sdesc(g.bsm + buf * kBBuf + q * kBMat, kNB * 16, 128);
                        asm volatile("{\n\t.reg .pred p;\n\tsetp.ne.b32 p, %4, 0;\n\t"
                                     "tcgen05.mma.cta_group::1.kind::f16 [%0], [%1], %2, %3, p;\n\t}"
                                     ::"r"(g.tD + buf * 32), "r"(g.tA + buf * 64 + 8 * q), "l"(db), "r"(idesc),
                                       "r"(q)
                                     : "memory");
                    }
                    asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];"
                                 ::"r"(g.bar + 8 * buf) : "memory");
                }
                // (2) epilogue of unit u - 1 while the tensor cores run unit u
                if (u > 0) {
                    const int pu = uc - 1;
                    mbar_wait(g.bar + 8 * (pu & 1), (pu >> 1) & 1, alive);
                    asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
                    epilogue<FMT>(prev, u - 1, g.tD + (pu & 1) * 32 + g.lane_off, ntok, st, acc);
                }
                prev = R[b].sc;
                ++uc;
            }
            // (3) refill this register slot
            const int sn = s + NB;
            if (sn < n_steps) {
                load_step<FMT>(P, sn, R[b]);
#pragma unroll
                for (int gg = 0; gg < G; ++gg)
                    if (xsrc) XB[b][gg] = ldg128(xsrc + (size_t)128 * (sn * G + gg));
            }
        }
    }
    // epilogue of the last unit; afterwards every MMA of this tensor has completed
    const int pu = uc - 1;
    mbar_wait(g.bar + 8 * (pu & 1), (pu >> 1) & 1, alive);
    asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
    epilogue<FMT>(prev, n_units - 1, g.tD + (pu & 1) * 32 + g.lane_off, ntok, st, acc);
    asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
}

struct TItem { int p, rb, ntok, shared; int vec[kDecodeTok], asg[kDecodeTok]; };

// item id -> (slot, 128-row block, token group); ids of a group only increase
template <bool kDown>
__device__ __forceinline__ void t_decode(const TArgs& A, const TSlots& sl, const int32_t* s_perm, int n_slots, int id,
                                         int& cursor, TItem& it) {
    while (cursor + 1 < n_slots && sl.pre[cursor + 1] <= id) ++cursor;
    const int p = cursor, local = id - sl.pre[p];
    const Dims& d = A.d;
    const int nrb = (kDown ? d.H : d.I) / kRowsT;
    const int tg = local / nrb;
    it.p = p;
    it.rb = local - tg * nrb;
    it.shared = p < d.has_shared;
    it.ntok = min(kDecodeTok, sl.ntot[p] - tg * kDecodeTok);
#pragma unroll
    for (int j = 0; j < kDecodeTok; ++j) {
        int t = 0, a = 0;
        if (j < it.ntok) {
            const int q = tg * kDecodeTok + j;
            if (it.shared) { t = q; a = d.T * d.K + q; }
            else {
                const int idx = sl.first[p] + q;
                a = idx < kMaxCachedAssign ? s_perm[idx] : A.perm[idx];
                t = a / d.K;
            }
        }
        it.asg[j] = a;
        it.vec[j] = kDown ? a : t;
    }
}

template <bool kDown>
__global__ void __launch_bounds__(kTThreads, 1) tgemv_kernel(const __grid_constant__ ExpertTab tab,
                                                             const __grid_constant__ TArgs A) {
    pdl_wait();
    pdl_launch();
    __shared__ TSlots sl;
    __shared__ int32_t s_perm[kMaxCachedAssign];
    __shared__ __align__(1024) uint8_t bmat[2][2][kBBuf];   // [group][buffer]
    __shared__ float xch[kRowsT][kDecodeTok];                // up sums handed to the gate group
    __shared__ __align__(8) uint64_t bars[2][2];            // [group][buffer]
    __shared__ uint32_t s_tmem;
    const Dims& d = A.d;
    const int tid = threadIdx.x, warp = tid >> 5;
    const int grp = warp >> 2, r = tid & 127;
    const int n_rb = (kDown ? d.H : d.I) / kRowsT;
    const int n_slots = A.active[0] + d.has_shared;
    for (int i = tid; i < n_slots; i += kTThreads) {
        int e;
        if (i < d.has_shared) { e = d.E; sl.first[i] = 0; sl.ntot[i] = d.T; }
        else {
            e = A.active[1 + i - d.has_shared];
            sl.first[i] = A.offsets[e]; sl.ntot[i] = A.offsets[e + 1] - A.offsets[e];
        }
        sl.ptr[i][0] = tab.p[e][kDown ? 2 : 0];
        sl.ptr[i][1] = tab.p[e][1];
        sl.fmt[i][0] = tab.fmt[e][kDown ? 2 : 0];
        sl.fmt[i][1] = tab.fmt[e][1];
        sl.down_fmt[i] = tab.fmt[e][2];
    }
    const int n_routed = min(d.T * d.K, kMaxCachedAssign);
    for (int i = tid; i < n_routed; i += kTThreads) s_perm[i] = A.perm[i];
    __syncthreads();
    if (tid == 0) {
        int run = 0;
        for (int i = 0; i < n_slots; ++i) {
            sl.pre[i] = run;
            run += n_rb * ((sl.ntot[i] + kDecodeTok - 1) / kDecodeTok);
        }
        sl.pre[n_slots] = run;
        for (int i = 0; i < 4; ++i)
            asm volatile("mbarrier.init.shared::cta.b64 [%0], 1;"
                         ::"r"((uint32_t)__cvta_generic_to_shared(&bars[0][0]) + 8 * i) : "memory");
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    }
    if (warp == 0) {
        asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;"
                     ::"r"((uint32_t)__cvta_generic_to_shared(&s_tmem)), "r"(512) : "memory");
        asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
    }
    asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
    __syncthreads();
    asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
    const uint32_t tbase = s_tmem;
    GCtx g;
    // group g: A buffers at columns 256 g + {0, 64}, D buffers at 256 g + 128 + {0, 32}
    g.tA = tbase + 256 * grp;
    g.tD = tbase + 256 * grp + 128;
    g.bsm = (uint32_t)__cvta_generic_to_shared(&bmat[grp][0][0]);
    g.bar = (uint32_t)__cvta_generic_to_shared(&bars[grp][0]);
    g.lane_off = (uint32_t)(32 * (warp & 3)) << 16;
    g.grp = grp;
    g.leader = r == 0;
    const int n_items = sl.pre[n_slots];
    const int nsb = kDown ? A.nsbi : A.nsbx;
    const __half* vq = kDown ? A.hq : A.xq;
    const float* vs = kDown ? A.hs : A.xs;
    const size_t q_stride = (size_t)kFamSlots * nsb * 256, s_stride = (size_t)nsb * kStatFloats;
    int cursor = 0, uc = 0, last_fmt = -1;
    bool ok = true, alive = true;
    // gate/up: both groups take the same item (gate rows, up rows); down: one item per group
    const int step = kDown ? 2 * gridDim.x : gridDim.x;
    const int first = kDown ? 2 * blockIdx.x + grp : blockIdx.x;
    for (int id = first; id < n_items && ok; id += step) {
        TItem it;
        t_decode<kDown>(A, sl, s_perm, n_slots, id, cursor, it);
        const int ph = kDown ? 0 : grp;   // tensor of this group: gate / up, or down
        const int fmt = sl.fmt[it.p][ph];
        const int64_t R = (int64_t)it.rb * kRowsT + r;
        const RowP P = row_planes(fmt, sl.ptr[it.p][ph], kDown ? d.H : d.I, kDown ? d.I : d.H, R);
        const float* st[kDecodeTok];
#pragma unroll
        for (int tk = 0; tk < kDecodeTok; ++tk) st[tk] = vs + (size_t)it.vec[tk < it.ntok ? tk : 0] * s_stride;
        // this thread's B slice: token r >> 4, positions 8 (r & 15) .. + 7 of each unit
        const __half* xsrc = nullptr;
        int boff = 0;
        if (r < 16 * it.ntok) {
            const int tk = r >> 4, c8 = r & 15, q = c8 >> 1;
            int v = it.vec[0];
#pragma unroll
            for (int j = 1; j < kDecodeTok; ++j) if (tk == j) v = it.vec[j];
            xsrc = vq + (size_t)v * q_stride + (size_t)tfam(fmt) * nsb * 256 + 8 * c8;
            const int n = (fmt == kQ2K || fmt == kQ3K) ? 8 * tk + q : 4 * tk + (q >> 1);
            boff = q * kBMat + ((c8 & 1) * kNB + n) * 16;
        }
        if (fmt != last_fmt) {
            // the zero pattern of the B matrices depends on the format; all MMAs
            // of this group have completed (end of run_tensor)
            for (int i = r; i < 2 * kBBuf / 16; i += 128)
                reinterpret_cast<uint4*>(&bmat[grp][0][0])[i] = make_uint4(0u, 0u, 0u, 0u);
            group_sync(grp);
            last_fmt = fmt;
        }
        float acc[kDecodeTok] = {0.0f, 0.0f, 0.0f, 0.0f};
        const int n_units = 2 * nsb;
        switch (fmt) {
        case kQ2K: run_tensor<kQ2K>(g, P, n_units, it.ntok, xsrc, boff, st, uc, alive, acc); break;
        case kQ3K: run_tensor<kQ3K>(g, P, n_units, it.ntok, xsrc, boff, st, uc, alive, acc); break;
        case kQ4K: run_tensor<kQ4K>(g, P, n_units, it.ntok, xsrc, boff, st, uc, alive, acc); break;
        default: run_tensor<kQ80>(g, P, n_units, it.ntok, xsrc, boff, st, uc, alive, acc); break;
        }
        if (kDown) {
#pragma unroll
            for (int tk = 0; tk < kDecodeTok; ++tk)
                if (tk < it.ntok) A.pdn[(size_t)it.asg[tk] * d.H + R] = acc[tk];
            ok = !group_any(grp, !alive);
        } else {
            // SwiGLU (routing weight folded in) and the prepared h of the down
            // projection; warp w of the gate group owns rows 32 w .. 32 w + 31
            if (grp == 1) {
#pragma unroll
                for (int tk = 0; tk < kDecodeTok; ++tk) xch[r][tk] = acc[tk];
            }
            __syncthreads();
            if (grp == 0) {
                const int famd = 1 << tfam(sl.down_fmt[it.p]);
                const int jb = (int)(R >> 5);
                const int n32 = d.I / 32;
#pragma unroll
                for (int tk = 0; tk < kDecodeTok; ++tk) {
                    if (tk >= it.ntok) break;
                    const int a = it.asg[tk];
                    const float gv = acc[tk];
                    const float w = it.shared ? 1.0f : A.wts[a];
                    const float hv = gv / (1.0f + expf(-gv)) * xch[r][tk] * w;
                    __half* hq = A.hq + (size_t)a * kFamSlots * A.nsbi * 256;
                    float* hs = A.hs + (size_t)a * A.nsbi * kStatFloats;
                    prep_block32(hv, jb, famd, hq, hs, A.nsbi);
                    if (jb == n32 - 1)
                        for (int jb2 = n32; jb2 < 8 * A.nsbi; ++jb2) prep_block32(0.0f, jb2, famd, hq, hs, A.nsbi);
                }
            }
            ok = !__syncthreads_or(!alive);
        }
    }
    if (!ok && r == 0) atomicOr(A.err, kErrT);
    // every MMA of the CTA has completed (each commit was waited for, or a
    // wait gave up and the error is recorded) before tensor memory is freed
    asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
    __syncthreads();
    if (warp == 0) {
        asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
        asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tbase), "r"(512) : "memory");
    }
}

}  // namespace

bool decode_tc_fits(const Dims& d) { return d.H % kRowsT == 0 && d.I % kRowsT == 0; }

cudaError_t launch_decode_tc(const Dims& d, const ExpertTab& tab, const Work& w, float* out, cudaStream_t s) {
    if (d.T == 0) return cudaSuccess;
    const int g_tsms = device_setup(kSetupTgemv, nullptr);
    if (g_tsms <= 0) return cudaErrorInvalidDevice;
    TArgs A;
    A.d = d;
    A.nsbx = (d.H + 255) / 256;
    A.nsbi = (d.I + 255) / 256;
    A.xq = w.xq; A.xs = w.xs; A.hq = w.hq; A.hs = w.hs;
    A.offsets = w.offsets; A.perm = w.perm; A.active = w.active; A.wts = w.wts;
    A.pdn = w.pdn; A.err = w.err;
    prof_begin("gateup_tgemv", s);
    cudaError_t err = launch_pdl(tgemv_kernel<false>, dim3(g_tsms), dim3(kTThreads), 0, s, tab, A);
    prof_end(s);
    if (err != cudaSuccess) return err;
    prof_begin("down_tgemv", s);
    err = launch_pdl(tgemv_kernel<true>, dim3(g_tsms), dim3(kTThreads), 0, s, tab, A);
    prof_end(s);
    if (err != cudaSuccess) return err;
    return launch_combine(d, w.pdn, out, s);
}

}  // namespace mq
