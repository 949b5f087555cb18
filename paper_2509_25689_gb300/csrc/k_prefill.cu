// Expert FFN for prefill-sized batches: a grouped GEMM per expert on the
// 5th-generation tensor cores (arXiv 2509.25689 Fig. 1 layer; expert tensors
// in their own k-quant style formats, Sec. 3.3).
//
// Work unit = (expert slot, 128 weight rows, up to 256 of the slot's tokens).
// The MMA is tcgen05.mma.cta_group::1.kind::f16 with M = 128 weight rows,
// N = the unit's tokens (rounded up to 16) and K in steps of 16, fp32
// accumulators in tensor memory (gate and up side by side for gate/up units).
// Per 64-wide K chunk the CTA's 128 threads dequantize their weight row of
// each tensor straight from the packed planes into fp16 (one row per thread,
// fp16 keeps 11 significant bits of the decoded weight), and gather the
// unit's activation rows (fp16 tokens, or the fp16 SwiGLU output h) with
// cp.async into a 3-slot ring; thread 0 issues the MMAs of a chunk and
// commits them to that slot's mbarrier while the threads prepare the next
// chunks.  Operands sit in shared memory in the canonical K-major layout
// without swizzle: 8 x 8 fp16 core matrices, 16 bytes per row, rows of a core
// matrix contiguous, core matrices 128 bytes apart along M/N and
// (rows x 16) bytes apart along K.
// Epilogue (tcgen05.ld, lane = weight row): gate/up -> h = silu(g) * u * w
// stored as fp16 per assignment; down -> one fp32 partial output row block
// per assignment, summed in slot order by the combine kernel.  Range: token
// t enters as fp16(x * 2^-e_t), e_t = the exponent of its largest |x| (so
// any finite bf16 token fits), and h as fp16(h * 2^-2 e_t); the epilogues
// undo both scalings in fp32.  An h that would still overflow fp16 sets an
// error bit (MQ_EDEVICE from moe_quant_status) instead of passing an inf on.
// Every mbarrier wait is bounded (about 1 s) and reports to the error word;
// tensor memory is released on every exit path.
#include <cuda_fp16.h>

#include "mq_internal.h"

namespace mq {
namespace {

constexpr int kPWorkers = 256;                 // 8 worker warps: two per TMEM lane quarter
constexpr int kMmaWarp = kPWorkers / 32;       // the down GEMM: + one warp that issues the MMAs
// The gate/up GEMM keeps the MMA issue in worker thread 0: at 9 warps a
// thread gets at most 168 registers, and its two tensors' prefetched fields
// spill there (2.57 -> 2.83 ms measured), while the down GEMM gains (1.97 ->
// 1.72 ms).
__host__ __device__ constexpr bool mma_warp(bool down) { return down; }
__host__ __device__ constexpr int prefill_threads(bool down) { return kPWorkers + (mma_warp(down) ? 32 : 0); }
constexpr int kMT = 128;                       // weight rows per unit (MMA M)
constexpr int kNT = 256;                       // tokens per unit (largest MMA N)
constexpr int kKC = 64;                        // K per ring slot
constexpr int kPSlots = 3;
constexpr int kABytes = kMT * kKC * 2;         // one weight chunk, 16 KB
constexpr int kBBytes = kNT * kKC * 2;         // one activation chunk, 32 KB
constexpr int kSlotBytes = 2 * kABytes + kBBytes;
constexpr uint32_t kErrMma = 4u;
constexpr uint32_t kErrRange = 16u;            // an fp16 SwiGLU output would overflow (see the epilogue)
constexpr uint32_t kErrWeightRange = 64u;      // a BF16 weight beyond the fp16 operand range

struct PrefillArgs {
    Dims d;
    const int32_t* offsets; const int32_t* perm; const int32_t* active; const float* wts;
    const __half* x16;       // [T][H] tokens in fp16, token t scaled by 2^-xe[t]
    const int32_t* xe;       // [T] the tokens' exponents
    __half* h16;             // [A][I] SwiGLU outputs (routing weight folded in), scaled by 2^-2 xe[t]
    float* pdn;              // [A][H]
    uint32_t* next;          // unit counters (gate/up, down), zeroed per call
    uint32_t* err;
};

struct PSlots {
    int32_t first[kMaxExperts + 1], ntot[kMaxExperts + 1], pre[kMaxExperts + 2];
    const uint8_t* ptr[kMaxExperts + 1][2];
    uint8_t fmt[kMaxExperts + 1][2];
};

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
__device__ __forceinline__ bool mbar_wait(uint32_t bar, uint32_t parity) {
    if (mbar_try(bar, parity)) return true;
    const uint64_t t0 = global_ns();
    for (;;) {
        if (mbar_try(bar, parity)) return true;
        if (global_ns() - t0 > 1000000000ull) return false;
    }
}
__device__ __forceinline__ void mbar_arrive(uint32_t bar) {
    asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(bar) : "memory");
}
// barrier 1 over the worker warps only (the MMA warp runs its own loop)
__device__ __forceinline__ void workers_sync() { asm volatile("bar.sync 1, %0;" ::"n"(kPWorkers) : "memory"); }
__device__ __forceinline__ bool workers_any(bool v) {
    uint32_t r;
    asm volatile("{\n\t.reg .pred p, q;\n\tsetp.ne.u32 p, %1, 0;\n\tbar.red.or.pred q, 1, %2, p;\n\tselp.u32 %0, 1, 0, q;\n\t}"
                 : "=r"(r) : "r"((uint32_t)v), "n"(kPWorkers) : "memory");
    return r != 0;
}
__device__ __forceinline__ uint64_t sdesc(uint32_t saddr, uint32_t lbo, uint32_t sbo) {
    return (uint64_t)((saddr & 0x3FFFFu) >> 4) | ((uint64_t)((lbo >> 4) & 0x3FFFu) << 16) |
           ((uint64_t)((sbo >> 4) & 0x3FFFu) << 32) | ((uint64_t)1 << 46);
}
// kind::f16 instruction descriptor: fp16 A and B, fp32 D, both K-major
__device__ __forceinline__ uint32_t idesc_f16(int M, int N) {
    return (1u << 4) | ((uint32_t)(N >> 3) << 17) | ((uint32_t)(M >> 4) << 24);
}
__device__ __forceinline__ void mma_f16(uint32_t dtmem, uint64_t da, uint64_t db, uint32_t idesc, uint32_t acc) {
    asm volatile("{\n\t.reg .pred p;\n\tsetp.ne.b32 p, %4, 0;\n\t"
                 "tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n\t}"
                 ::"r"(dtmem), "l"(da), "l"(db), "r"(idesc), "r"(acc) : "memory");
}
__device__ __forceinline__ void sts128(uint32_t a, uint32_t x, uint32_t y, uint32_t z, uint32_t w) {
    asm volatile("st.shared.v4.u32 [%0], {%1,%2,%3,%4};" ::"r"(a), "r"(x), "r"(y), "r"(z), "r"(w) : "memory");
}
__device__ __forceinline__ uint32_t h2u(__half2 h) { return *reinterpret_cast<uint32_t*>(&h); }
__device__ __forceinline__ __half2 u2h(uint32_t u) { return *reinterpret_cast<__half2*>(&u); }
__device__ __forceinline__ uint32_t ldg32(const uint8_t* p) { return __ldg(reinterpret_cast<const unsigned int*>(p)); }
__device__ __forceinline__ uint4 ldg128(const uint8_t* p) { return __ldg(reinterpret_cast<const uint4*>(p)); }
__device__ __forceinline__ uint32_t sub4(uint4 v, int i) { return i == 0 ? v.x : i == 1 ? v.y : i == 2 ? v.z : v.w; }

// fp16 pair "1024 + c" for the two codes at bit offset s of each 16-bit half
__device__ __forceinline__ __half2 code_pair(uint32_t w, int s, uint32_t mask) {
    return u2h(((w >> s) & mask) | 0x64006400u);
}

// Raw packed fields of one weight row for one 64-wide chunk of the
// contraction, loaded one chunk ahead of their use.
struct Packed {
    uint32_t w[16];   // code words (Q8_0: two blocks x 8; Q4_K: two sub-blocks x 4; Q2_K/Q3_K: 4 low + 4 high)
    uint32_t sc[4];   // scale record (Q2_K 16 B, Q3_K / Q4_K 12 B)
    uint32_t dd;      // d | dmin << 16 (Q8_0: d of the two blocks)
};

__device__ __forceinline__ uint2 ldg64u(const uint8_t* p) { return __ldg(reinterpret_cast<const uint2*>(p)); }
__device__ __forceinline__ uint32_t ldg16u(const uint8_t* p) { return __ldg(reinterpret_cast<const unsigned short*>(p)); }

// Start of one weight row's records in each plane; the record of
// superblock (Q8_0: block) b is at row[p] + b * 32 * record_bytes[p].
struct RowPtrs {
    const uint8_t* row[4];
};
__device__ __forceinline__ RowPtrs row_ptrs(int fmt, const uint8_t* base, const TensorLayout& L, int64_t R) {
    RowPtrs P;
    const PlaneBytes pb = plane_bytes(fmt);
#pragma unroll
    for (int p = 0; p < 4; ++p) P.row[p] = p < pb.n ? rec_ptr(base + L.plane[p], L, pb.b[p], R, 0) : nullptr;
    return P;
}

// kRare: the launch's layer has Q6_K or BF16 tensors (their code paths exist
// only in that instantiation, so the common one keeps its registers)
template <bool kRare>
__device__ __forceinline__ void load_chunk(int fmt, const RowPtrs& RP, int c, int hf, Packed& P) {
    if (kRare && fmt == kBF16) {
        // block 2c + hf: only the address of its 64-byte record is carried (the
        // decode step loads it), which keeps the prefetched fields of the other
        // formats in registers
        const uintptr_t bp = reinterpret_cast<uintptr_t>(RP.row[0] + (int64_t)(2 * c + hf) * (32 * 64));
        P.w[0] = (uint32_t)bp;
        P.w[1] = (uint32_t)((uint64_t)bp >> 32);
        return;
    }
    if (fmt == kQ80) {
        const int64_t b = 2 * c + hf;
        const uint8_t* cp = RP.row[1] + b * (32 * 32);
        const uint4 w0 = ldg128(cp), w1 = ldg128(cp + 16);
        P.w[0] = w0.x; P.w[1] = w0.y; P.w[2] = w0.z; P.w[3] = w0.w;
        P.w[4] = w1.x; P.w[5] = w1.y; P.w[6] = w1.z; P.w[7] = w1.w;
        P.dd = ldg16u(RP.row[0] + b * (32 * 2));
        return;
    }
    const int64_t s = c >> 2;
    const int cc = c & 3;
    P.dd = ldg16u(RP.row[0] + s * (32 * 2));
    if (fmt == kQ4K) {
        P.dd |= ldg16u(RP.row[1] + s * (32 * 2)) << 16;
        const uint8_t* sp = RP.row[2] + s * (32 * 12);
        P.sc[0] = ldg32(sp); P.sc[1] = ldg32(sp + 4); P.sc[2] = ldg32(sp + 8);
        const int j = 2 * cc + hf;
        const uint4 w = ldg128(RP.row[3] + s * (32 * 128) + (j >> 2) * (kRowTile * 64) + 16 * (j & 3));
        P.w[0] = w.x; P.w[1] = w.y; P.w[2] = w.z; P.w[3] = w.w;
        return;
    }
    if (kRare && fmt == kQ6K) {
        const uint4 sv = ldg128(RP.row[1] + s * (32 * 16));
        P.sc[0] = sv.x; P.sc[1] = sv.y; P.sc[2] = sv.z; P.sc[3] = sv.w;
        // low nibbles: sub-block j = 4 cc + i in unit cc / 2, words 4 i + 2 (cc % 2) + 0..1
        const uint8_t* np = RP.row[2] + s * (32 * 128) + (cc >> 1) * (kRowTile * 64);
        const uint8_t* hp = RP.row[3] + s * (32 * 64);
#pragma unroll
        for (int ii = 0; ii < 2; ++ii) {
            const int i = 2 * hf + ii;
            const uint2 nw = ldg64u(np + 4 * (4 * i + 2 * (cc & 1)));
            P.w[2 * ii] = nw.x; P.w[2 * ii + 1] = nw.y;
            P.w[4 + ii] = ldg32(hp + 4 * (4 * i + cc));
        }
        return;
    }
    if (fmt == kQ2K) {
        P.dd |= ldg16u(RP.row[1] + s * (32 * 2)) << 16;
        const uint4 sv = ldg128(RP.row[2] + s * (32 * 16));
        P.sc[0] = sv.x; P.sc[1] = sv.y; P.sc[2] = sv.z; P.sc[3] = sv.w;
        const uint8_t* cp = RP.row[3] + s * (32 * 64);
#pragma unroll
        for (int ii = 0; ii < 2; ++ii) { const int i = 2 * hf + ii; P.w[ii] = ldg32(cp + 4 * (4 * i + cc)); }
        return;
    }
    // Q3_K
    const uint8_t* sp = RP.row[1] + s * (32 * 12);
    P.sc[0] = ldg32(sp); P.sc[1] = ldg32(sp + 4); P.sc[2] = ldg32(sp + 8);
    const uint8_t* lp = RP.row[2] + s * (32 * 64);
    const uint8_t* hp = RP.row[3] + s * (32 * 32);
#pragma unroll
    for (int ii = 0; ii < 2; ++ii) {
        const int i = 2 * hf + ii;
        P.w[ii] = ldg32(lp + 4 * (4 * i + cc));
        P.w[4 + ii] = ldg32(hp + 4 * (2 * i + (cc >> 1)));
    }
}

// One superblock's packed fields of one weight row for this thread's half of
// each of its four 64-wide chunks (Q2_K, Q3_K, Q4_K): codes, scales and d /
// dmin are read once per superblock, with wide loads, one superblock ahead.
struct SBlk {
    uint4 cw[4];      // Q2_K / Q3_K low bits: words 4i..4i+3 for i = 2 hf, 2 hf + 1; Q4_K: the 4 chunks' 16 bytes
    uint2 hw[2];      // Q3_K high bits: words 2i, 2i+1
    uint32_t sc[4];   // scale record
    uint32_t dd;      // d | dmin << 16
};
__device__ __forceinline__ void load_sblk(int fmt, const RowPtrs& RP, int sb, int hf, SBlk& B) {
    const int64_t s = sb;
    B.dd = ldg16u(RP.row[0] + s * (32 * 2));
    if (fmt == kQ4K) {
        B.dd |= ldg16u(RP.row[1] + s * (32 * 2)) << 16;
        const uint8_t* sp = RP.row[2] + s * (32 * 12);
        B.sc[0] = ldg32(sp); B.sc[1] = ldg32(sp + 4); B.sc[2] = ldg32(sp + 8);
#pragma unroll
        for (int cc = 0; cc < 4; ++cc) {
            const int j = 2 * cc + hf;
            B.cw[cc] = ldg128(RP.row[3] + s * (32 * 128) + (j >> 2) * (kRowTile * 64) + 16 * (j & 3));
        }
    } else if (fmt == kQ2K) {
        B.dd |= ldg16u(RP.row[1] + s * (32 * 2)) << 16;
        const uint4 sv = ldg128(RP.row[2] + s * (32 * 16));
        B.sc[0] = sv.x; B.sc[1] = sv.y; B.sc[2] = sv.z; B.sc[3] = sv.w;
#pragma unroll
        for (int ii = 0; ii < 2; ++ii) B.cw[ii] = ldg128(RP.row[3] + s * (32 * 64) + 16 * (2 * hf + ii));
    } else {   // Q3_K
        const uint8_t* sp = RP.row[1] + s * (32 * 12);
        B.sc[0] = ldg32(sp); B.sc[1] = ldg32(sp + 4); B.sc[2] = ldg32(sp + 8);
#pragma unroll
        for (int ii = 0; ii < 2; ++ii) {
            B.cw[ii] = ldg128(RP.row[2] + s * (32 * 64) + 16 * (2 * hf + ii));
            B.hw[ii] = ldg64u(RP.row[3] + s * (32 * 32) + 8 * (2 * hf + ii));
        }
    }
}
// the chunk's fields (chunk cc of the superblock) in the per-chunk form dequant_store reads
__device__ __forceinline__ void make_packed(int fmt, const SBlk& B, int cc, Packed& P) {
    P.dd = B.dd;
#pragma unroll
    for (int i = 0; i < 4; ++i) P.sc[i] = B.sc[i];
    if (fmt == kQ4K) {
        P.w[0] = B.cw[cc].x; P.w[1] = B.cw[cc].y; P.w[2] = B.cw[cc].z; P.w[3] = B.cw[cc].w;
    } else {
#pragma unroll
        for (int ii = 0; ii < 2; ++ii) {
            P.w[ii] = sub4(B.cw[ii], cc);
            P.w[4 + ii] = (cc >> 1) ? B.hw[ii].y : B.hw[ii].x;
        }
    }
}

__device__ __forceinline__ float half_lo(uint32_t v) { return __half2float(__ushort_as_half((unsigned short)(v & 0xffffu))); }
__device__ __forceinline__ float half_hi(uint32_t v) { return __half2float(__ushort_as_half((unsigned short)(v >> 16))); }
// byte i (0..15) of a 4-word record, with a runtime i kept in registers
__device__ __forceinline__ uint32_t byte_of(const uint32_t (&w)[4], int i) {
    const int k = i >> 2;
    const uint32_t v = k == 0 ? w[0] : k == 1 ? w[1] : k == 2 ? w[2] : w[3];
    return (v >> (8 * (i & 3))) & 0xffu;
}

// Q6_K and BF16 chunks, kept out of line: the formats of most units keep
// their registers (an out-of-line call saves only what is live around it).
// The fields come as scalars (a reference would make every caller keep its
// packed fields in local memory).
__device__ __noinline__ bool dequant_store_rare(int fmt, uint32_t w0, uint32_t w1, uint32_t w2, uint32_t w3,
                                                uint32_t w4, uint32_t w5, uint32_t sc0, uint32_t sc1, uint32_t sc2,
                                                uint32_t sc3, uint32_t dd, int c, int hf, uint32_t dst) {
    const uint32_t Pw[6] = {w0, w1, w2, w3, w4, w5};
    const uint32_t Psc[4] = {sc0, sc1, sc2, sc3};
    if (fmt == kBF16) {
        const uint8_t* bp = reinterpret_cast<const uint8_t*>((uintptr_t)w0 | ((uintptr_t)w1 << 32));
        uint32_t wd[16];   // the record: pair p of the block in word 4 (p % 4) + p / 4
#pragma unroll
        for (int v = 0; v < 4; ++v) {
            const uint4 q = ldg128(bp + 16 * v);
            wd[4 * v] = q.x; wd[4 * v + 1] = q.y; wd[4 * v + 2] = q.z; wd[4 * v + 3] = q.w;
        }
        bool over = false;
#pragma unroll
        for (int q = 0; q < 4; ++q) {   // core-matrix row 4 hf + q: k = 8q .. 8q+7 of the block
            uint32_t o[4];
#pragma unroll
            for (int pp = 0; pp < 4; ++pp) {
                const uint32_t wv = wd[4 * pp + q];   // the pair k = 8q + 2pp, +1
                const float lo = __uint_as_float(wv << 16), hi = __uint_as_float(wv & 0xFFFF0000u);
                over |= fmaxf(fabsf(lo), fabsf(hi)) >= 65520.0f;
                o[pp] = h2u(__floats2half2_rn(lo, hi));
            }
            sts128(dst + ((4 * hf + q) * kMT) * 16, o[0], o[1], o[2], o[3]);
        }
        return over;
    }
    if (fmt == kQ6K) {
        const int cc = c & 3;
        const float d = half_lo(dd);
        const __half2 k1056 = __float2half2_rn(1056.0f);   // 1024 + the code offset 32
#pragma unroll
        for (int ii = 0; ii < 2; ++ii) {
            const int i = 2 * hf + ii, j = 4 * cc + i;
            const int sv = (int)byte_of(Psc, q16_slot(j)) - 128;
            const __half2 a2 = __float2half2_rn(d * (float)sv);
#pragma unroll
            for (int q = 0; q < 2; ++q) {
                uint32_t o[4];
#pragma unroll
                for (int mm = 0; mm < 4; ++mm) {
                    const int m = 4 * q + mm;
                    const uint32_t nib = (Pw[2 * ii + (m >> 2)] >> (4 * (m & 3))) & 0x000F000Fu;
                    const uint32_t hi2 = (Pw[4 + ii] >> (2 * m)) & 0x00030003u;
                    o[mm] = h2u(__hmul2(a2, __hsub2(u2h(nib | (hi2 << 4) | 0x64006400u), k1056)));
                }
                sts128(dst + ((2 * i + q) * kMT) * 16, o[0], o[1], o[2], o[3]);
            }
        }
        return false;
    }
    return false;
}

// Decode the 64 weights of chunk c of one row (fields in P) to fp16 and store
// them as 8 core-matrix rows at dst, dst + 128*16, ...  Values follow the
// format definitions of include/moeq.h; the per-sub-block products d*sc and
// dmin*m are rounded to fp16 once.  BF16 weights convert exactly where
// 2^-14 <= |w| < 65520 (below, to the nearest fp16 subnormal); the return
// value is true if one of them is beyond the fp16 range.
template <bool kRare>
__device__ __forceinline__ bool dequant_store(int fmt, const Packed& P, int c, int hf, uint32_t dst) {
    const __half2 k1024 = __float2half2_rn(1024.0f);
    if (kRare && (fmt == kBF16 || fmt == kQ6K))
        return dequant_store_rare(fmt, P.w[0], P.w[1], P.w[2], P.w[3], P.w[4], P.w[5], P.sc[0], P.sc[1], P.sc[2],
                                  P.sc[3], P.dd, c, hf, dst);
    if (fmt == kQ80) {
        const __half2 k1152 = __float2half2_rn(1152.0f);
        {
            const int bb = hf;
            const __half2 d2 = __float2half2_rn(half_lo(P.dd));
#pragma unroll
            for (int q = 0; q < 4; ++q) {   // core-matrix row kc = 4 bb + q: pairs m = 4q .. 4q+3
                uint32_t o[4];
#pragma unroll
                for (int mm = 0; mm < 4; ++mm) {
                    const int m = 4 * q + mm;
                    o[mm] = h2u(__hmul2(d2, __hsub2(code_pair(P.w[m >> 1], 8 * (m & 1), 0x00FF00FFu), k1152)));
                }
                sts128(dst + ((4 * bb + q) * kMT) * 16, o[0], o[1], o[2], o[3]);
            }
        }
        return false;
    }
    const int cc = c & 3;
    const float d = half_lo(P.dd);
    if (fmt == kQ4K) {
        const float dmin = half_hi(P.dd);
        {
            const int jj = hf, j = 2 * cc + jj;
            const uint32_t lo = byte_of(P.sc, j), high = P.sc[2] >> (4 * j);
            const int sc = (int)(lo & 15u) | (int)((high & 3u) << 4), mn = (int)(lo >> 4) | (int)(((high >> 2) & 3u) << 4);
            const __half2 a2 = __float2half2_rn(d * (float)sc), nb2 = __float2half2_rn(-(dmin * (float)mn));
#pragma unroll
            for (int q = 0; q < 4; ++q) {
                uint32_t o[4];
#pragma unroll
                for (int mm = 0; mm < 4; ++mm) {
                    const int m = 4 * q + mm;
                    o[mm] = h2u(__hfma2(a2, __hsub2(code_pair(P.w[m >> 2], 4 * (m & 3), 0x000F000Fu), k1024), nb2));
                }
                sts128(dst + ((4 * jj + q) * kMT) * 16, o[0], o[1], o[2], o[3]);
            }
        }
        return false;
    }
    if (fmt == kQ2K) {
        const float dmin = half_hi(P.dd);
#pragma unroll
        for (int ii = 0; ii < 2; ++ii) {
            const int i = 2 * hf + ii, j = 4 * cc + i;
            const uint32_t f = byte_of(P.sc, q16_slot(j));
            const __half2 a2 = __float2half2_rn(d * (float)(f & 15u)), nb2 = __float2half2_rn(-(dmin * (float)(f >> 4)));
#pragma unroll
            for (int q = 0; q < 2; ++q) {
                uint32_t o[4];
#pragma unroll
                for (int mm = 0; mm < 4; ++mm) {
                    const int m = 4 * q + mm;
                    o[mm] = h2u(__hfma2(a2, __hsub2(code_pair(P.w[ii], 2 * m, 0x00030003u), k1024), nb2));
                }
                sts128(dst + ((2 * i + q) * kMT) * 16, o[0], o[1], o[2], o[3]);
            }
        }
        return false;
    }
    // Q3_K
    const __half2 k1028 = __float2half2_rn(1028.0f);
#pragma unroll
    for (int ii = 0; ii < 2; ++ii) {
        const int i = 2 * hf + ii, j = 4 * cc + i;
        const int u = q16_slot(j);
        const int sfield = (int)((byte_of(P.sc, u >> 1) >> (4 * (u & 1))) & 15u) |
                           (int)(((byte_of(P.sc, 8 + (u >> 2)) >> (2 * (u & 3))) & 3u) << 4);
        const __half2 a2 = __float2half2_rn(d * (float)(sfield - 32));
        const uint32_t wl = P.w[ii], wh = P.w[4 + ii] >> (8 * (cc & 1));
#pragma unroll
        for (int q = 0; q < 2; ++q) {
            uint32_t o[4];
#pragma unroll
            for (int mm = 0; mm < 4; ++mm) {
                const int m = 4 * q + mm;
                const uint32_t t = ((wl >> (2 * m)) & 0x00030003u) | (((wh >> m) & 0x00010001u) << 2) | 0x64006400u;
                o[mm] = h2u(__hmul2(a2, __hsub2(u2h(t), k1028)));
            }
            sts128(dst + ((2 * i + q) * kMT) * 16, o[0], o[1], o[2], o[3]);
        }
    }
    return false;
}

__device__ __forceinline__ float silu(float v) { return v / (1.0f + expf(-v)); }

template <bool kDown, bool kRare>
__global__ void __launch_bounds__(prefill_threads(kDown), 1) prefill_kernel(const __grid_constant__ ExpertTab tab,
                                                                            const __grid_constant__ PrefillArgs A) {
    constexpr bool kWS = mma_warp(kDown);
    constexpr int kPThreads = prefill_threads(kDown);
    pdl_wait();
    pdl_launch();
    extern __shared__ __align__(1024) uint8_t smem[];
    __shared__ PSlots sl;
    __shared__ int32_t s_row[kNT], s_asg[kNT], s_ex[kNT];
    __shared__ float s_w[kNT];
    __shared__ __align__(8) uint64_t bars[kPSlots];   // the MMAs of the slot's chunk are done
    __shared__ __align__(8) uint64_t fbar[kPSlots];   // the slot's chunk is in shared memory (every worker)
    __shared__ int s_info[kPSlots];                   // that chunk: N rounded to 16 | accumulate << 16, or -1 = end
    __shared__ uint32_t s_tmem;
    __shared__ int s_fail;
    __shared__ int s_unit;
    const Dims& d = A.d;
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int n_mt = (kDown ? d.H : d.I) / kMT;
    const int K = kDown ? d.I : d.H;
    const int n_slots = A.active[0] + d.has_shared;
    // slot table: shared expert first, then the active routed experts
    for (int i = tid; i < n_slots; i += kPThreads) {
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
    }
    __syncthreads();
    if (tid == 0) {
        int run = 0;
        for (int i = 0; i < n_slots; ++i) { sl.pre[i] = run; run += n_mt * ((sl.ntot[i] + kNT - 1) / kNT); }
        sl.pre[n_slots] = run;
        s_fail = 0;
        for (int i = 0; i < kPSlots; ++i) {
            asm volatile("mbarrier.init.shared::cta.b64 [%0], 1;" ::"r"((uint32_t)__cvta_generic_to_shared(&bars[i]))
                         : "memory");
            asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;"
                         ::"r"((uint32_t)__cvta_generic_to_shared(&fbar[i])), "n"(kPWorkers) : "memory");
        }
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    }
    constexpr int kCols = kDown ? 256 : 512;
    if (warp == 0) {
        asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;"
                     ::"r"((uint32_t)__cvta_generic_to_shared(&s_tmem)), "r"(kCols) : "memory");
        asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
    }
    asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
    __syncthreads();
    asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
    const uint32_t tbase = s_tmem;
    const uint32_t ring = (uint32_t)__cvta_generic_to_shared(smem);
    const uint32_t bar0 = (uint32_t)__cvta_generic_to_shared(bars);
    const uint32_t fbar0 = (uint32_t)__cvta_generic_to_shared(fbar);
    const int n_units = sl.pre[n_slots];
    const int nC = K / kKC;
    // the MMAs of the chunk in ring slot s (info: N rounded to 16 | accumulate << 16),
    // committed to the slot's barrier, which frees the slot
    auto issue_chunk = [&](int s, int info) {
        asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
        const uint32_t idesc = idesc_f16(kMT, info & 0xffff);
        const uint32_t sbase = ring + s * kSlotBytes, bsm = sbase + 2 * kABytes;
#pragma unroll
        for (int ks = 0; ks < kKC / 16; ++ks) {
            const uint32_t acc = ((info >> 16) != 0 || ks > 0) ? 1u : 0u;
            const uint64_t db = sdesc(bsm + 2 * ks * kNT * 16, kNT * 16, 128);
            mma_f16(tbase, sdesc(sbase + 2 * ks * kMT * 16, kMT * 16, 128), db, idesc, acc);
            if (!kDown) mma_f16(tbase + kNT, sdesc(sbase + kABytes + 2 * ks * kMT * 16, kMT * 16, 128), db, idesc, acc);
        }
        asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];"
                     ::"r"(bar0 + 8 * s) : "memory");
    };

    if (kWS && warp == kMmaWarp) {
        // ---- MMA issue: the CTA's chunk g sits in ring slot g % kPSlots once
        // every worker has arrived on its full barrier; one lane issues its
        // MMAs and commits them to the slot's barrier (which frees the slot)
        int last = -1;
        bool ok = true;
        for (int g = 0;; ++g) {
            const int s = g % kPSlots;
            if (!mbar_wait(fbar0 + 8 * s, (g / kPSlots) & 1)) { ok = false; break; }
            const int info = s_info[s];
            if (info < 0) break;
            if (lane == 0) issue_chunk(s, info);
            __syncwarp();
            last = g;
        }
        if (!ok && lane == 0) { atomicOr(A.err, kErrMma); s_fail = 1; }
        // tensor memory is released only after the MMAs issued here are done
        if (last >= 0) mbar_wait(bar0 + 8 * (last % kPSlots), (last / kPSlots) & 1);
    } else {
    int gchunk = 0;        // chunks posted by this CTA so far (ring position and parities)
    int last_committed = -1;   // without the MMA warp: the last chunk thread 0 committed
    bool failed = false;
    bool w_over = false;   // a BF16 weight of this thread's rows beyond the fp16 range
    int cursor = 0;

    // units are claimed from a global counter (their cost varies with the
    // number of tokens of the expert, up to 16x between full and small tiles)
    for (;;) {
        if (tid == 0) s_unit = (int)atomicAdd(A.next + (kDown ? 1 : 0), 1u);
        workers_sync();
        const int u = s_unit;
        if (u >= n_units || failed) break;
        while (cursor + 1 < n_slots && sl.pre[cursor + 1] <= u) ++cursor;
        const int p = cursor, local = u - sl.pre[p];
        const int tt = local / n_mt, mt = local - tt * n_mt;
        const int n0 = tt * kNT, N = min(kNT, sl.ntot[p] - n0), Npad = (N + 15) & ~15;
        const bool shared = p < d.has_shared;
        // the unit's activation rows, assignments and weights
        for (int n = tid; n < kNT; n += kPWorkers) {
            int a = -1, row = 0, ex = 0;
            float w = 0.0f;
            if (n < N) {
                const int q = n0 + n;
                if (shared) { a = d.T * d.K + q; row = q; w = 1.0f; }
                else { a = A.perm[sl.first[p] + q]; row = a / d.K; w = A.wts[a]; }
                ex = A.xe[row];   // row is the token here
                if (kDown) row = a;
            }
            s_row[n] = row; s_asg[n] = a; s_w[n] = w; s_ex[n] = ex;
        }
        const int f0 = sl.fmt[p][0], f1 = sl.fmt[p][1];
        const TensorLayout L0 = tensor_layout(f0, kDown ? d.H : d.I, K);
        const TensorLayout L1 = tensor_layout(f1, d.I, K);
        const uint8_t* b0 = sl.ptr[p][0];
        const uint8_t* b1 = sl.ptr[p][1];
        const int rr = tid & (kMT - 1), hf = tid >> 7;   // weight row of the unit, half of each chunk
        const int64_t R = (int64_t)mt * kMT + rr;
        const RowPtrs RP0 = row_ptrs(f0, b0, L0, R);
        const RowPtrs RP1 = kDown ? RP0 : row_ptrs(f1, b1, L1, R);
        workers_sync();
        // B gather: this thread always moves the 16-byte piece kc = tid % 8 of
        // rows n = tid / 8 + 32 j; the row pointers are fixed for the unit
        const __half* src = kDown ? A.h16 : A.x16;
        const int kcg = tid & 7, n_base = tid >> 3;
        const __half* gsrc[kNT / 32];
#pragma unroll
        for (int j = 0; j < kNT / 32; ++j) {
            const int n = n_base + 32 * j;
            gsrc[j] = n < N ? src + (size_t)s_row[n] * K + kcg * 8 : nullptr;
        }
        auto gather = [&](int c, int s) {
            const uint32_t bdst = ring + s * kSlotBytes + 2 * kABytes + (kcg * kNT + n_base) * 16;
#pragma unroll
            for (int j = 0; j < kNT / 32; ++j) {
                const int n = n_base + 32 * j;
                if (n >= Npad) break;
                const uint32_t dst = bdst + 32 * j * 16;
                if (gsrc[j] != nullptr)
                    asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(dst), "l"(gsrc[j] + c * kKC) : "memory");
                else
                    sts128(dst, 0u, 0u, 0u, 0u);
            }
        };
        gather(0, gchunk % kPSlots);
        asm volatile("cp.async.commit_group;" ::: "memory");
        // L2 prefetch duty: lanes 0..7 of warps 0..3 (the unit's four 32-row
        // tiles): lane = plane (0..3) of tensor lane / 4; a superblock's records
        // of a tile are one contiguous range per plane
        const uint8_t* pf_src = nullptr;
        uint32_t pf_bytes = 0;
        int pf_nsb = 0;   // whole superblocks of records a row has (Q8_0: groups of 8 blocks)
        if (hf == 0 && lane < 8 && (!kDown || lane < 4)) {
            const int pl = lane & 3, fmt = lane < 4 ? f0 : f1;
            const PlaneBytes pb = plane_bytes(fmt);
            if (pl < pb.n) {
                const TensorLayout& Lx = lane < 4 ? L0 : L1;
                pf_src = rec_ptr((lane < 4 ? b0 : b1) + Lx.plane[pl], Lx, pb.b[pl], (int64_t)mt * kMT + 32 * warp, 0);
                const bool b32 = block_len(fmt) == 32;   // Q8_0 / BF16: groups of 8 blocks
                pf_bytes = (uint32_t)(32 * pb.b[pl] * (b32 ? 8 : 1));
                pf_nsb = (int)(b32 ? Lx.blocks_per_row / 8 : Lx.blocks_per_row);
                if ((reinterpret_cast<uintptr_t>(pf_src) & 15u) != 0 || (pf_bytes & 15u) != 0) pf_src = nullptr;
            }
        }
        // one 64-wide chunk: gather the next chunk's rows, decode this one's
        // weights, then post the chunk to the MMA warp (no block barrier: the
        // workers run ahead up to the ring's depth) or, without it, meet at a
        // barrier after which thread 0 issues the chunk's MMAs
        auto chunk_body = [&](int c, const Packed& Q0, const Packed& Q1) -> bool {
            const int g = gchunk + c, s = g % kPSlots;
            bool bad = false;
            if (c + 1 < nC) {
                const int g1 = g + 1, s1 = g1 % kPSlots;
                // slot s1 was last used by chunk g1 - kPSlots: its MMAs must be done
                if (g1 >= kPSlots) bad = !mbar_wait(bar0 + 8 * s1, ((g1 - kPSlots) / kPSlots) & 1);
                if (!bad) gather(c + 1, s1);
            }
            asm volatile("cp.async.commit_group;" ::: "memory");
            const uint32_t sbase = ring + s * kSlotBytes;
            if (dequant_store<kRare>(f0, Q0, c, hf, sbase + rr * 16)) w_over = true;
            if (!kDown && dequant_store<kRare>(f1, Q1, c, hf, sbase + kABytes + rr * 16)) w_over = true;
            asm volatile("cp.async.wait_group 1;" ::: "memory");
            // this thread's shared-memory writes (and landed copies) before the
            // tensor cores read them
            asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
            const int info = Npad | (c > 0 ? 1 << 16 : 0);
            if (kWS) {
                if (tid == 0) s_info[s] = info;
                mbar_arrive(fbar0 + 8 * s);
                if (bad) s_fail = 1;   // checked by all workers at the unit's end
                return true;
            }
            if (workers_any(bad)) return false;
            if (tid == 0) issue_chunk(s, info);
            last_committed = g;
            return true;
        };
        auto sblk_fmt = [](int f) { return f == kQ2K || f == kQ3K || f == kQ4K; };
        if (sblk_fmt(f0) && (kDown || sblk_fmt(f1))) {
            // superblock-granular fields (Q2_K, Q3_K, Q4_K), one superblock ahead
            const int nS = (nC + 3) / 4;
            SBlk Sa0, Sa1, Sb0, Sb1;
            load_sblk(f0, RP0, 0, hf, Sa0);
            if (!kDown) load_sblk(f1, RP1, 0, hf, Sa1);
            auto sblock = [&](int sb, const SBlk& C0, const SBlk& C1, SBlk& N0, SBlk& N1) -> bool {
                if (sb + 1 < nS) {
                    load_sblk(f0, RP0, sb + 1, hf, N0);
                    if (!kDown) load_sblk(f1, RP1, sb + 1, hf, N1);
                }
                // the records of the superblock after that into L2
                if (pf_src != nullptr && sb + 2 < pf_nsb)
                    asm volatile("cp.async.bulk.prefetch.L2.global [%0], %1;"
                                 ::"l"(pf_src + (int64_t)(sb + 2) * pf_bytes), "r"(pf_bytes) : "memory");
#pragma unroll
                for (int cc = 0; cc < 4; ++cc) {
                    const int c = 4 * sb + cc;
                    if (c >= nC) break;
                    Packed Q0, Q1;
                    make_packed(f0, C0, cc, Q0);
                    if (!kDown) make_packed(f1, C1, cc, Q1);
                    if (!chunk_body(c, Q0, Q1)) return false;
                }
                return true;
            };
            for (int sb = 0; sb < nS; sb += 2) {
                if (!sblock(sb, Sa0, Sa1, Sb0, Sb1)) { failed = true; break; }
                if (sb + 1 < nS && !sblock(sb + 1, Sb0, Sb1, Sa0, Sa1)) { failed = true; break; }
            }
        } else {
            // Q8_0, Q6_K or BF16 in the unit: per-chunk fields, one chunk ahead
            Packed P0, P1;                 // this chunk's packed fields, gate (or down) and up
            load_chunk<kRare>(f0, RP0, 0, hf, P0);
            if (!kDown) load_chunk<kRare>(f1, RP1, 0, hf, P1);
            for (int c = 0; c < nC; ++c) {
                // pull the records of this warp's 32-row tile for the next superblock
                // into L2, so the per-thread loads of the coming chunks hit L2
                if ((c & 3) == 0 && pf_src != nullptr && (c >> 2) + 1 < pf_nsb)
                    asm volatile("cp.async.bulk.prefetch.L2.global [%0], %1;"
                                 ::"l"(pf_src + (int64_t)((c >> 2) + 1) * pf_bytes), "r"(pf_bytes) : "memory");
                Packed N0, N1;             // the next chunk's, loaded while this one is decoded
                if (c + 1 < nC) {
                    load_chunk<kRare>(f0, RP0, c + 1, hf, N0);
                    if (!kDown) load_chunk<kRare>(f1, RP1, c + 1, hf, N1);
                }
                if (!chunk_body(c, P0, P1)) { failed = true; break; }
                P0 = N0;
                if (!kDown) P1 = N1;
            }
        }
        asm volatile("cp.async.wait_group 0;" ::: "memory");
        if (failed) break;
        // all MMAs of the unit are done once the last chunk's commit arrived
        const int glast = gchunk + nC - 1;
        const bool ok = mbar_wait(bar0 + 8 * (glast % kPSlots), (glast / kPSlots) & 1);
        if (workers_any(!ok || s_fail)) { failed = true; break; }
        gchunk += nC;
        asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
        // epilogue: TMEM lane 32 warp + lane = weight row, columns = tokens
        const int quarter = warp & 3;
        const int row = mt * kMT + 32 * quarter + lane;
        for (int n = 8 * (warp >> 2); n < Npad; n += 16) {
            uint32_t g8[8], u8[8];
            const uint32_t ta = tbase + ((uint32_t)(32 * quarter) << 16) + (uint32_t)n;
            asm volatile("tcgen05.ld.sync.aligned.32x32b.x8.b32 {%0,%1,%2,%3,%4,%5,%6,%7}, [%8];"
                         : "=r"(g8[0]), "=r"(g8[1]), "=r"(g8[2]), "=r"(g8[3]), "=r"(g8[4]), "=r"(g8[5]), "=r"(g8[6]),
                           "=r"(g8[7]) : "r"(ta));
            if (!kDown)
                asm volatile("tcgen05.ld.sync.aligned.32x32b.x8.b32 {%0,%1,%2,%3,%4,%5,%6,%7}, [%8];"
                             : "=r"(u8[0]), "=r"(u8[1]), "=r"(u8[2]), "=r"(u8[3]), "=r"(u8[4]), "=r"(u8[5]),
                               "=r"(u8[6]), "=r"(u8[7]) : "r"(ta + kNT));
            asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
            // tokens enter scaled by 2^-e (e = s_ex): gate and up sums are
            // multiplied back before SwiGLU, h leaves scaled by 2^-2e (it
            // grows like the square of the token), the down sums are
            // multiplied back by 2^2e
            bool over = false;
#pragma unroll
            for (int j = 0; j < 8; ++j) {
                const int nn = n + j;
                if (nn >= N) break;
                const int a = s_asg[nn], ex = s_ex[nn];
                if (kDown) {
                    A.pdn[(size_t)a * d.H + row] = ldexpf(__uint_as_float(g8[j]), 2 * ex);
                } else {
                    const float gv = ldexpf(__uint_as_float(g8[j]), ex), uv = ldexpf(__uint_as_float(u8[j]), ex);
                    const float hs = ldexpf(silu(gv) * uv * s_w[nn], -2 * ex);
                    over |= !(fabsf(hs) <= 65504.0f);
                    A.h16[(size_t)a * d.I + row] = __float2half_rn(hs);
                }
            }
            if (over) atomicOr(A.err, kErrRange);
        }
        // the accumulators are read: the next unit's MMAs (posted after this
        // point by every worker) may overwrite them
        asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
        workers_sync();
    }
    if (failed) {
        if (tid == 0) { atomicOr(A.err, kErrMma); s_fail = 1; }
        // wait (bounded) for the MMAs still in flight before giving TMEM back
        if (!kWS && last_committed >= 0)
            mbar_wait(bar0 + 8 * (last_committed % kPSlots), (last_committed / kPSlots) & 1);
    } else if (kWS) {
        // end marker for the MMA warp in the next chunk's slot (every earlier
        // chunk's MMAs are done, so the warp has read every earlier marker)
        const int s = gchunk % kPSlots;
        if (tid == 0) s_info[s] = -1;
        mbar_arrive(fbar0 + 8 * s);
    }
    if (w_over) atomicOr(A.err, kErrWeightRange);
    }   // workers
    __syncthreads();
    asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
    __syncthreads();
    if (warp == 0) {
        asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
        asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tbase), "r"(kCols) : "memory");
    }
}

void prefill_setup() {
    const int smem = kPSlots * kSlotBytes;
    cudaFuncSetAttribute(prefill_kernel<false, false>, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
    cudaFuncSetAttribute(prefill_kernel<true, false>, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
    cudaFuncSetAttribute(prefill_kernel<false, true>, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
    cudaFuncSetAttribute(prefill_kernel<true, true>, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
}

}  // namespace

cudaError_t launch_prefill(const Dims& d, const ExpertTab& tab, const Work& w, float* out, cudaStream_t s) {
    if (d.T == 0) return cudaSuccess;
    const int smem = kPSlots * kSlotBytes;
    const int g_psms = device_setup(kSetupPrefill, prefill_setup);
    if (g_psms <= 0) return cudaErrorInvalidDevice;
    PrefillArgs A;
    A.d = d;
    A.offsets = w.offsets; A.perm = w.perm; A.active = w.active; A.wts = w.wts;
    A.x16 = w.x16; A.xe = w.xe; A.h16 = w.h16; A.pdn = w.pdn; A.err = w.err;
    A.next = w.counters;
    bool rare = false;   // a Q6_K or BF16 tensor anywhere in the layer
    for (int e = 0; e < d.E + d.has_shared; ++e)
        for (int j = 0; j < 3; ++j) rare |= tab.fmt[e][j] == kQ6K || tab.fmt[e][j] == kBF16;
    prof_begin("gateup_tc", s);
    cudaError_t err = rare ? launch_pdl(prefill_kernel<false, true>, dim3(g_psms), dim3(prefill_threads(false)), smem,
                                        s, tab, A)
                           : launch_pdl(prefill_kernel<false, false>, dim3(g_psms), dim3(prefill_threads(false)), smem,
                                        s, tab, A);
    prof_end(s);
    if (err != cudaSuccess) return err;
    prof_begin("down_tc", s);
    err = rare ? launch_pdl(prefill_kernel<true, true>, dim3(g_psms), dim3(prefill_threads(true)), smem, s, tab, A)
               : launch_pdl(prefill_kernel<true, false>, dim3(g_psms), dim3(prefill_threads(true)), smem, s, tab, A);
    prof_end(s);
    if (err != cudaSuccess) return err;
    return launch_combine(d, w.pdn, out, s);
}

}  // namespace mq
