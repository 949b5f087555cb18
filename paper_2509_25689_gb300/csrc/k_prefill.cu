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
    uint8_t* xp;             // warp-specialised GEMM: the tokens in slot-position order, tiled (shares pdn's bytes)
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
    for (int i = 0; i < 32; ++i)
        if (mbar_try(bar, parity)) return true;
    const uint64_t t0 = global_ns();
    for (;;) {
        for (int i = 0; i < 32; ++i)
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

// ---------------------------------------------------------------------------
// Warp-specialised form of the same GEMM, for layers whose tensors are all
// Q2_K, Q3_K, Q4_K or Q8_0.  Each CTA runs four roles at once, so that the
// record loads, the weight decode, the activation gather and the MMAs of
// different chunks overlap instead of following one another:
//   - a producer warp claims the units, publishes each one (slot, rows,
//     tokens) in a two-deep unit ring and streams the unit's packed records
//     into a two-stage ring with bulk copies (one per tensor, plane and
//     32-row tile; a stage holds one superblock, or 128 contraction columns
//     when a tensor is Q8_0, whose K-quant partner then comes twice);
//   - sixteen worker warps decode the records from shared memory into the
//     fp16 operand of each 64-wide chunk (the values dequant_store gives;
//     gate/up: eight warps per tensor, down: eight per chunk parity) and, at
//     the unit's end, run the epilogue out of tensor memory; the gate/up
//     epilogue writes h straight into the down GEMM's activation layout;
//   - an activation warp moves the chunk's activation rows with eight bulk
//     copies from the tile-ordered copy of the tokens (xperm_kernel) or of h;
//   - an MMA warp issues a chunk's MMAs once the workers and the activation
//     warp have filled its operand slot (a two-slot ring) and commits them
//     to the slot's empty barrier.
// Every wait is bounded and reports to the error word.
// 16 worker warps (gate/up: 8 per tensor; down: 8 per chunk parity), then
// the producer, activation and MMA warps
__host__ __device__ constexpr int g_workers(bool down) { return 16; }
__host__ __device__ constexpr int g_threads(bool down) { return (g_workers(down) + 3) * 32; }
constexpr int kGNT = 256;                      // tokens per unit (MMA N up to 256)
// operand slots: gate/up two of A gate | A up | B (64 KB), down three of
// A | B (48 KB); a third gate/up slot fits only with 128-token units,
// measured slower on the Zipf prefill
__host__ __device__ constexpr int g_ops(bool down) { return down ? 3 : 2; }
__host__ __device__ constexpr int g_bofs(bool down) { return down ? kABytes : 2 * kABytes; }
__host__ __device__ constexpr int g_slot(bool down) { return g_bofs(down) + kGNT * kKC * 2; }
constexpr int kGOpsMax = 3;
constexpr int kGPk = 2;                        // packed-record stages
constexpr int kGPkBytes = 36 * 1024;           // Q4_K + Q4_K superblock of 128 rows: 2 x 18,432
__host__ __device__ constexpr int g_smem(bool down) { return g_ops(down) * g_slot(down) + kGPk * kGPkBytes; }

// Activation rows of the warp-specialised GEMM in the order its units read
// them: slot positions r (the permutation's order for the routed experts,
// T*K + t for the shared expert), cut into tiles of up to kGNT rows of one
// slot.  In a tile of N rows starting at position r0, the 16-byte piece p
// (columns 8p .. 8p+7) of row n sits (p * N + n) * 16 bytes after r0 * K * 2,
// so a 64-column chunk of a tile is eight contiguous runs of N x 16 bytes:
// one bulk copy each into the canonical operand layout.
__device__ __forceinline__ size_t perm_piece(int r0, int K, int N, int p, int n) {
    return (size_t)r0 * K * 2 + ((size_t)p * N + n) * 16;
}

// The tokens (fp16, as the logits kernel scaled them) in that layout.  Work
// items are (tile, 64 pieces) of the call's tiles (the slots' tiles in slot
// order); warp w writes the runs of pieces w, w + 8, ... of its item: lane l
// the rows l, l + 32, ... of a run, so every store of a warp is 512
// contiguous bytes.
constexpr int kXpWarps = 8, kXpPieces = 64;
__global__ void __launch_bounds__(kXpWarps * 32) xperm_kernel(const __half* __restrict__ x16,
                                                              const int32_t* __restrict__ offsets,
                                                              const int32_t* __restrict__ perm,
                                                              const int32_t* __restrict__ active, const Dims d,
                                                              uint8_t* __restrict__ xp) {
    pdl_wait();
    __shared__ int32_t s_first[kMaxExperts + 1], s_ntot[kMaxExperts + 1], s_pre[kMaxExperts + 2];
    __shared__ int32_t s_tok[kGNT];
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int n_slots = active[0] + d.has_shared, TK = d.T * d.K, np = d.H / 8;
    for (int i = tid; i < n_slots; i += blockDim.x) {
        if (i < d.has_shared) { s_first[i] = TK; s_ntot[i] = d.T; }
        else {
            const int e = active[1 + i - d.has_shared];
            s_first[i] = offsets[e]; s_ntot[i] = offsets[e + 1] - offsets[e];
        }
    }
    __syncthreads();
    if (tid == 0) {
        int run = 0;
        for (int i = 0; i < n_slots; ++i) { s_pre[i] = run; run += (s_ntot[i] + kGNT - 1) / kGNT; }
        s_pre[n_slots] = run;
    }
    __syncthreads();
    // work items: (tile, block of kXpPieces pieces), so that large tiles spread over CTAs
    const int n_pb = (np + kXpPieces - 1) / kXpPieces, n_items = s_pre[n_slots] * n_pb;
    int p = 0;
    for (int it = blockIdx.x; it < n_items; it += gridDim.x) {
        const int ti = it / n_pb, pb = it - ti * n_pb;
        while (p + 1 < n_slots && s_pre[p + 1] <= ti) ++p;
        const int tt = ti - s_pre[p], r0 = s_first[p] + tt * kGNT, N = min(kGNT, s_ntot[p] - tt * kGNT);
        __syncthreads();   // the previous item's token ids are read
        for (int n = tid; n < N; n += blockDim.x) s_tok[n] = p < d.has_shared ? tt * kGNT + n : perm[r0 + n] / d.K;
        __syncthreads();
        uint8_t* dst = xp + (size_t)r0 * d.H * 2;
        const int pe = min(np, (pb + 1) * kXpPieces);
        for (int pc = pb * kXpPieces + warp; pc < pe; pc += kXpWarps) {
            uint4 v[kGNT / 32];   // all loads of the run first, then the stores
#pragma unroll
            for (int j = 0; j < kGNT / 32; ++j) {
                const int n = lane + 32 * j;
                if (n < N) v[j] = __ldg(reinterpret_cast<const uint4*>(x16 + (size_t)s_tok[n] * d.H) + pc);
            }
#pragma unroll
            for (int j = 0; j < kGNT / 32; ++j) {
                const int n = lane + 32 * j;
                if (n < N) *reinterpret_cast<uint4*>(dst + ((size_t)pc * N + n) * 16) = v[j];
            }
        }
    }
    pdl_launch();
}

// per-CTA slot table of the warp-specialised GEMM (the pointers come from
// the expert table by the slot's expert id)
struct GSlots {
    int32_t first[kMaxExperts + 1], ntot[kMaxExperts + 1], pre[kMaxExperts + 2], e[kMaxExperts + 1];
    uint8_t fmt[kMaxExperts + 1][2];
};

struct GUnit {
    int u;               // unit id, -1 once there are none left
    int p, mt, N, Npad;
    int r0;              // the tile's first slot position
    int ks;              // contraction columns per packed stage: 256, or 128 when a tensor is Q8_0
};

// where each plane of each tensor sits in a packed stage (tile 0; tile t at + t * tile)
struct GStage {
    int off[2][4], tile[2][4], ub[2][4];
    int total;
};
__device__ __forceinline__ GStage gstage(int f0, int f1, int ntens, int ks) {
    GStage G;
    int at = 0;
#pragma unroll
    for (int z = 0; z < 2; ++z) {
        const int f = z == 0 ? f0 : f1;
        const PlaneBytes pb = plane_bytes(f);
        const int nb = f == kQ80 ? ks / 32 : 1;
#pragma unroll
        for (int pl = 0; pl < 4; ++pl) {
            const bool on = z < ntens && pl < pb.n;
            G.off[z][pl] = at;
            G.tile[z][pl] = on ? nb * 32 * pb.b[pl] : 0;
            G.ub[z][pl] = on ? unit_bytes(pb.b[pl]) : 0;
            at += 4 * G.tile[z][pl];
        }
    }
    G.total = at;
    return G;
}

__device__ __forceinline__ void g_mbar_init(uint32_t bar, uint32_t count) {
    asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(bar), "r"(count) : "memory");
}
__device__ __forceinline__ void g_arrive_tx(uint32_t bar, uint32_t bytes) {
    asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(bar), "r"(bytes) : "memory");
}
__device__ __forceinline__ void g_bulk(uint32_t dst, const void* src, uint32_t bytes, uint32_t bar, uint64_t pol) {
    asm volatile("cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes.L2::cache_hint [%0], [%1], %2, [%3], %4;"
                 ::"r"(dst), "l"(src), "r"(bytes), "r"(bar), "l"(pol) : "memory");
}
__device__ __forceinline__ uint4 g_lds128(uint32_t a) {
    uint4 v;
    asm volatile("ld.shared.v4.u32 {%0,%1,%2,%3}, [%4];" : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w) : "r"(a));
    return v;
}
__device__ __forceinline__ uint2 g_lds64(uint32_t a) {
    uint2 v;
    asm volatile("ld.shared.v2.u32 {%0,%1}, [%2];" : "=r"(v.x), "=r"(v.y) : "r"(a));
    return v;
}
__device__ __forceinline__ uint32_t g_lds32(uint32_t a) {
    uint32_t v;
    asm volatile("ld.shared.u32 %0, [%1];" : "=r"(v) : "r"(a));
    return v;
}
__device__ __forceinline__ uint32_t g_lds16(uint32_t a) {
    unsigned short v;
    asm volatile("ld.shared.u16 %0, [%1];" : "=h"(v) : "r"(a));
    return v;
}

// One superblock's fields of this thread's row (records at rec[pl] in the
// stage), as load_sblk reads them from global memory.
__device__ __forceinline__ void load_sblk_s(int fmt, const uint32_t (&rec)[4], int hf, SBlk& B) {
    B.dd = g_lds16(rec[0]);
    if (fmt == kQ4K) {
        B.dd |= g_lds16(rec[1]) << 16;
        B.sc[0] = g_lds32(rec[2]); B.sc[1] = g_lds32(rec[2] + 4); B.sc[2] = g_lds32(rec[2] + 8);
#pragma unroll
        for (int cc = 0; cc < 4; ++cc) {
            const int j = 2 * cc + hf;
            B.cw[cc] = g_lds128(rec[3] + (j >> 2) * (kRowTile * 64) + 16 * (j & 3));
        }
    } else if (fmt == kQ2K) {
        B.dd |= g_lds16(rec[1]) << 16;
        const uint4 sv = g_lds128(rec[2]);
        B.sc[0] = sv.x; B.sc[1] = sv.y; B.sc[2] = sv.z; B.sc[3] = sv.w;
#pragma unroll
        for (int ii = 0; ii < 2; ++ii) B.cw[ii] = g_lds128(rec[3] + 16 * (2 * hf + ii));
    } else {   // Q3_K
        B.sc[0] = g_lds32(rec[1]); B.sc[1] = g_lds32(rec[1] + 4); B.sc[2] = g_lds32(rec[1] + 8);
#pragma unroll
        for (int ii = 0; ii < 2; ++ii) {
            B.cw[ii] = g_lds128(rec[2] + 16 * (2 * hf + ii));
            B.hw[ii] = g_lds64(rec[3] + 8 * (2 * hf + ii));
        }
    }
}
// make_packed for a chunk index known only at run time (selects instead of
// an indexed register array, which would live in local memory)
__device__ __forceinline__ uint4 pick4(const uint4 (&v)[4], int i) {
    const uint4 a = (i & 1) ? v[1] : v[0], b = (i & 1) ? v[3] : v[2];
    return (i & 2) ? b : a;
}
__device__ __forceinline__ void make_packed_rt(int fmt, const SBlk& B, int cc, Packed& P) {
    P.dd = B.dd;
#pragma unroll
    for (int i = 0; i < 4; ++i) P.sc[i] = B.sc[i];
    if (fmt == kQ4K) {
        const uint4 w = pick4(B.cw, cc);
        P.w[0] = w.x; P.w[1] = w.y; P.w[2] = w.z; P.w[3] = w.w;
    } else {
#pragma unroll
        for (int ii = 0; ii < 2; ++ii) {
            const uint4 w = B.cw[ii];
            const uint32_t lo = (cc & 1) ? w.y : w.x, hi = (cc & 1) ? w.w : w.z;
            P.w[ii] = (cc & 2) ? hi : lo;
            P.w[4 + ii] = (cc >> 1) ? B.hw[ii].y : B.hw[ii].x;
        }
    }
}
// Q8_0 block lb of the stage for this thread's row, as load_chunk reads it
__device__ __forceinline__ void load_q80_s(const uint32_t (&rec)[4], int lb, Packed& P) {
    const uint32_t cp = rec[1] + lb * (32 * 32);
    const uint4 w0 = g_lds128(cp), w1 = g_lds128(cp + 16);
    P.w[0] = w0.x; P.w[1] = w0.y; P.w[2] = w0.z; P.w[3] = w0.w;
    P.w[4] = w1.x; P.w[5] = w1.y; P.w[6] = w1.z; P.w[7] = w1.w;
    P.dd = g_lds16(rec[0] + lb * (32 * 2));
}

// ---- chunk decode for the warp-specialised GEMM: the values dequant_store
// produces (the same fp16 roundings: d * sc and dmin * m are exact products
// rounded once, then one fused multiply-add per weight pair), with fewer
// instructions: a code field at bit s <= 8 of each 16-bit half, OR-ed into
// the fp16 pair 2^(10 - s), reads as 2^(10 - s) + code exactly (the field
// lands in the mantissa at unit weight), so one AND-OR and one subtraction
// give the code without a shift; the scale fields of two sub-blocks are
// widened as one fp16 pair.  Stores are plain shared-memory stores the
// compiler may schedule (the proxy fence after them orders them for the
// tensor cores).
__device__ __forceinline__ constexpr uint32_t magic_bits(int s) {
    return ((uint32_t)(25 - s) << 10) | ((uint32_t)(25 - s) << 26);
}
__device__ __forceinline__ __half2 magic_val(int s) { return u2h(magic_bits(s)); }
__device__ __forceinline__ uint32_t pick_word(const uint32_t (&w)[4], int i) {
    const uint32_t a = (i & 1) ? w[1] : w[0], b = (i & 1) ? w[3] : w[2];
    return (i & 2) ? b : a;
}
__device__ __forceinline__ void st_row(uint4* dst, uint32_t a, uint32_t b, uint32_t c, uint32_t d) {
    *dst = make_uint4(a, b, c, d);
}

// Q2_K: sub-blocks 2 hf, 2 hf + 1 of chunk cc (16 weights each)
__device__ __forceinline__ void dq_q2k(const SBlk& B, int cc, int hf, uint4* dst) {
    const uint32_t dd = B.dd;
    const __half2 d2 = u2h((dd & 0xFFFFu) * 0x00010001u);
    const __half2 nm2 = u2h(((dd >> 16) * 0x00010001u) ^ 0x80008000u);   // -dmin
    const int s0 = q16_slot(4 * cc + 2 * hf);   // the two sub-blocks' slots: s0, s0 + 1 (s0 even)
    const uint32_t x = __byte_perm(pick_word(B.sc, s0 >> 2), 0u, (s0 & 2) ? 0x4342u : 0x4140u);
    const __half2 k1024 = magic_val(0);
    const __half2 scp = __hsub2(u2h((x & 0x000F000Fu) | 0x64006400u), k1024);
    const __half2 mp = __hsub2(u2h(((x >> 4) & 0x000F000Fu) | 0x64006400u), k1024);
    const __half2 ap = __hmul2(d2, scp), np = __hmul2(nm2, mp);
#pragma unroll
    for (int ii = 0; ii < 2; ++ii) {
        const int i = 2 * hf + ii;
        const __half2 a2 = ii ? __high2half2(ap) : __low2half2(ap);
        const __half2 n2 = ii ? __high2half2(np) : __low2half2(np);
        const uint4 cw = B.cw[ii];
        const uint32_t lo = (cc & 1) ? cw.y : cw.x, hi = (cc & 1) ? cw.w : cw.z;
        const uint32_t w = (cc & 2) ? hi : lo, wh = w >> 10;
        uint32_t o[8];
        o[0] = h2u(__hfma2(a2, __hsub2(u2h((w & 0x00030003u) | magic_bits(0)), magic_val(0)), n2));
        o[1] = h2u(__hfma2(a2, __hsub2(u2h((w & 0x000C000Cu) | magic_bits(2)), magic_val(2)), n2));
        o[2] = h2u(__hfma2(a2, __hsub2(u2h((w & 0x00300030u) | magic_bits(4)), magic_val(4)), n2));
        o[3] = h2u(__hfma2(a2, __hsub2(u2h((w & 0x00C000C0u) | magic_bits(6)), magic_val(6)), n2));
        o[4] = h2u(__hfma2(a2, __hsub2(u2h((w & 0x03000300u) | magic_bits(8)), magic_val(8)), n2));
        o[5] = h2u(__hfma2(a2, __hsub2(u2h((wh & 0x00030003u) | magic_bits(0)), magic_val(0)), n2));
        o[6] = h2u(__hfma2(a2, __hsub2(u2h((wh & 0x000C000Cu) | magic_bits(2)), magic_val(2)), n2));
        o[7] = h2u(__hfma2(a2, __hsub2(u2h((wh & 0x00300030u) | magic_bits(4)), magic_val(4)), n2));
        st_row(dst + (2 * i) * kMT, o[0], o[1], o[2], o[3]);
        st_row(dst + (2 * i + 1) * kMT, o[4], o[5], o[6], o[7]);
    }
}

// Q3_K: code q = low two bits + 4 * high bit, weight d * (s - 32) * (q - 4)
__device__ __forceinline__ void dq_q3k(const SBlk& B, int cc, int hf, uint4* dst) {
    const __half2 d2 = u2h((B.dd & 0xFFFFu) * 0x00010001u);
    const int u = q16_slot(4 * cc + 2 * hf);   // slots u, u + 1 (u even)
    const uint32_t lo = (pick_word(B.sc, u >> 3) >> (8 * ((u >> 1) & 3))) & 0xFFu;   // nibbles of slots u, u + 1
    const uint32_t hb = (B.sc[2] >> (8 * (u >> 2) + 2 * (u & 3))) & 0xFu;            // high bits: 2 per slot
    const uint32_t sx = (lo & 15u) | ((hb & 3u) << 4) | (((lo >> 4) | ((hb >> 2) << 4)) << 16);
    const __half2 ap = __hmul2(d2, __hsub2(u2h(sx | 0x64006400u), u2h(0x64206420u)));
    #pragma unroll
    for (int ii = 0; ii < 2; ++ii) {
        const int i = 2 * hf + ii;
        const __half2 a2 = ii ? __high2half2(ap) : __low2half2(ap);
        const uint4 cw = B.cw[ii];
        const uint32_t l0 = (cc & 1) ? cw.y : cw.x, l1 = (cc & 1) ? cw.w : cw.z;
        const uint32_t wl = (cc & 2) ? l1 : l0, wl8 = wl >> 8;
        const uint32_t wh = ((cc >> 1) ? B.hw[ii].y : B.hw[ii].x) >> (8 * (cc & 1));
        // pair m: low bits at 2m (m < 4) or 2m - 8 of wl >> 8 (m >= 4); its
        // high bit (bit m of wh) moved two bits above them
        uint32_t o[8];
#pragma unroll
        for (int m = 0; m < 8; ++m) {
            const int p = m < 4 ? 2 * m : 2 * m - 8;          // low bits' position
            const int sh = p + 2 - m;                          // high bit: m -> p + 2
            const uint32_t hsh = sh >= 0 ? (wh << sh) : (wh >> -sh);
            const uint32_t lm = 0x00030003u << p, hm = 0x00010001u << (p + 2);
            const uint32_t t = ((m < 4 ? wl : wl8) & lm) | (hsh & hm) | magic_bits(p);
            // (2^(10-p) + q) - (2^(10-p) + 4) = q - 4, exact
            o[m] = h2u(__hmul2(a2, __hsub2(u2h(t), u2h(magic_bits(p) + (4u << p) * 0x00010001u))));
        }
        st_row(dst + (2 * i) * kMT, o[0], o[1], o[2], o[3]);
        st_row(dst + (2 * i + 1) * kMT, o[4], o[5], o[6], o[7]);
    }
}

// Q4_K: sub-block j = 2 cc + hf (32 weights), weight d * sc * q - dmin * m
__device__ __forceinline__ void dq_q4k(const SBlk& B, int cc, int hf, uint4* dst) {
    const int j = 2 * cc + hf;
    const uint32_t lo = (pick_word(B.sc, j >> 2) >> (8 * (j & 3))) & 0xFFu, high = B.sc[2] >> (4 * j);
    const uint32_t sc = (lo & 15u) | ((high & 3u) << 4), mn = (lo >> 4) | (((high >> 2) & 3u) << 4);
    // (d, -dmin) * (sc, m): both products in one pair
    const __half2 dm = u2h((B.dd & 0xFFFFu) | ((B.dd & 0xFFFF0000u) ^ 0x80000000u));
    const __half2 pr = __hmul2(dm, __hsub2(u2h((sc | (mn << 16)) | 0x64006400u), magic_val(0)));
    const __half2 a2 = __low2half2(pr), n2 = __high2half2(pr);
    const uint4 cw = pick4(B.cw, cc);
    const uint32_t W[4] = {cw.x, cw.y, cw.z, cw.w};
#pragma unroll
    for (int q = 0; q < 4; ++q) {
        const uint32_t w = W[q], w8 = w >> 8;
        const uint32_t o0 = h2u(__hfma2(a2, __hsub2(u2h((w & 0x000F000Fu) | magic_bits(0)), magic_val(0)), n2));
        const uint32_t o1 = h2u(__hfma2(a2, __hsub2(u2h((w & 0x00F000F0u) | magic_bits(4)), magic_val(4)), n2));
        const uint32_t o2 = h2u(__hfma2(a2, __hsub2(u2h((w8 & 0x000F000Fu) | magic_bits(0)), magic_val(0)), n2));
        const uint32_t o3 = h2u(__hfma2(a2, __hsub2(u2h((w8 & 0x00F000F0u) | magic_bits(4)), magic_val(4)), n2));
        st_row(dst + (4 * hf + q) * kMT, o0, o1, o2, o3);
    }
}

// Q8_0: block 2 c + hf of the chunk (32 weights), weight d * (q - 128)
__device__ __forceinline__ void dq_q80(const uint32_t (&w)[8], uint32_t d16, int hf, uint4* dst) {
    const __half2 d2 = u2h((d16 & 0xFFFFu) * 0x00010001u);
    const __half2 k1152 = u2h(0x64806480u);   // 1024 + 128
#pragma unroll
    for (int q = 0; q < 4; ++q) {
        uint32_t o[4];
#pragma unroll
        for (int h = 0; h < 2; ++h) {
            const uint32_t v = w[2 * q + h];
            o[2 * h] = h2u(__hmul2(d2, __hsub2(u2h((v & 0x00FF00FFu) | 0x64006400u), k1152)));
            o[2 * h + 1] = h2u(__hmul2(d2, __hsub2(u2h(((v >> 8) & 0x00FF00FFu) | 0x64006400u), k1152)));
        }
        st_row(dst + (4 * hf + q) * kMT, o[0], o[1], o[2], o[3]);
    }
}

template <bool kDown>
__global__ void __launch_bounds__(g_threads(kDown), 1) gemm_ws_kernel(const __grid_constant__ ExpertTab tab,
                                                                      const __grid_constant__ PrefillArgs A) {
    constexpr int kTens = kDown ? 1 : 2;
    constexpr int kW = g_workers(kDown);            // worker warps
    constexpr int kThr = g_threads(kDown);
    constexpr int kWarpP = kW, kWarpB = kW + 1, kWarpM = kW + 2;
    constexpr int kGOps = g_ops(kDown), kGSlotBytes = g_slot(kDown), kBOfs = g_bofs(kDown);
    pdl_wait();
    pdl_launch();
    extern __shared__ __align__(1024) uint8_t smem[];
    __shared__ GSlots sl;
    __shared__ GUnit s_unit[2];
    __shared__ int32_t s_row[2][kGNT], s_asg[2][kGNT], s_ex[2][kGNT];
    __shared__ float s_w[2][kGNT];
    __shared__ __align__(8) uint64_t op_full[kGOpsMax], op_empty[kGOpsMax], pk_full[kGPk], pk_empty[kGPk];
    __shared__ __align__(8) uint64_t u_full[2], u_empty[2];
    __shared__ uint32_t s_tmem;
    __shared__ int s_fail;
    const Dims& d = A.d;
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int n_mt = (kDown ? d.H : d.I) / kMT;
    const int K = kDown ? d.I : d.H;
    const int nC = K / kKC;
    const int n_slots = A.active[0] + d.has_shared;
    for (int i = tid; i < n_slots; i += kThr) {
        int e;
        if (i < d.has_shared) { e = d.E; sl.first[i] = d.T * d.K; sl.ntot[i] = d.T; }
        else {
            e = A.active[1 + i - d.has_shared];
            sl.first[i] = A.offsets[e]; sl.ntot[i] = A.offsets[e + 1] - A.offsets[e];
        }
        sl.e[i] = e;
        sl.fmt[i][0] = tab.fmt[e][kDown ? 2 : 0];
        sl.fmt[i][1] = tab.fmt[e][1];
    }
    __syncthreads();
    const uint32_t ring = (uint32_t)__cvta_generic_to_shared(smem);
    const uint32_t pk0 = ring + kGOps * kGSlotBytes;
    const uint32_t opf = (uint32_t)__cvta_generic_to_shared(op_full), ope = (uint32_t)__cvta_generic_to_shared(op_empty);
    const uint32_t pkf = (uint32_t)__cvta_generic_to_shared(pk_full), pke = (uint32_t)__cvta_generic_to_shared(pk_empty);
    const uint32_t uf = (uint32_t)__cvta_generic_to_shared(u_full), ue = (uint32_t)__cvta_generic_to_shared(u_empty);
    if (tid == 0) {
        int run = 0;
        for (int i = 0; i < n_slots; ++i) { sl.pre[i] = run; run += n_mt * ((sl.ntot[i] + kGNT - 1) / kGNT); }
        sl.pre[n_slots] = run;
        s_fail = 0;
        // operand slot: the worker warps that decode a chunk (all 16 for
        // gate/up, 8 for down) and the activation warp's expect-tx arrival; packed stage and unit slot: one
        // arrival per worker warp (+ the activation and MMA warps)
        for (int i = 0; i < kGOps; ++i) { g_mbar_init(opf + 8 * i, 32 * (kDown ? kW / 2 : kW) + 1); g_mbar_init(ope + 8 * i, 1); }
        for (int i = 0; i < kGPk; ++i) { g_mbar_init(pkf + 8 * i, 1); g_mbar_init(pke + 8 * i, kW); }
        for (int i = 0; i < 2; ++i) { g_mbar_init(uf + 8 * i, 1); g_mbar_init(ue + 8 * i, kW + 2); }
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    }
    constexpr int kCols = kDown ? kGNT : 2 * kGNT;
    if (warp == 0) {
        asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;"
                     ::"r"((uint32_t)__cvta_generic_to_shared(&s_tmem)), "r"(kCols) : "memory");
        asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
    }
    asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
    __syncthreads();
    asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
    const uint32_t tbase = s_tmem;
    const int n_units = sl.pre[n_slots];
    auto failed = [&]() { return *reinterpret_cast<volatile int*>(&s_fail) != 0; };
    auto fail = [&]() { atomicOr(A.err, kErrMma); s_fail = 1; };

    if (warp == kWarpP) {
        // ---- producer: units and packed records
        const uint64_t pol = [] { uint64_t p; asm volatile("createpolicy.fractional.L2::evict_first.b64 %0, 1.0;" : "=l"(p)); return p; }();
        int cursor = 0, pq = 0;
        for (int ui = 0;; ++ui) {
            const int us = ui & 1;
            if (ui >= 2 && !mbar_wait(ue + 8 * us, ((ui - 2) >> 1) & 1)) { if (lane == 0) fail(); break; }
            int u = 0;
            if (lane == 0) u = (int)atomicAdd(A.next + (kDown ? 1 : 0), 1u);
            u = __shfl_sync(0xffffffffu, u, 0);
            if (u >= n_units || failed()) {
                if (lane == 0) { s_unit[us].u = -1; mbar_arrive(uf + 8 * us); }
                break;
            }
            while (cursor + 1 < n_slots && sl.pre[cursor + 1] <= u) ++cursor;
            const int p = cursor, local = u - sl.pre[p];
            const int tt = local / n_mt, mt = local - tt * n_mt;
            const int n0 = tt * kGNT, N = min(kGNT, sl.ntot[p] - n0);
            const bool shared = p < d.has_shared;
            for (int n = lane; n < kGNT; n += 32) {
                int a = -1, row = 0, ex = 0;
                float w = 0.0f;
                if (n < N) {
                    const int q = n0 + n;
                    if (shared) { a = d.T * d.K + q; row = q; w = 1.0f; }
                    else { a = A.perm[sl.first[p] + q]; row = a / d.K; w = A.wts[a]; }
                    ex = A.xe[row];
                    if (kDown) row = a;
                }
                s_row[us][n] = row; s_asg[us][n] = a; s_w[us][n] = w; s_ex[us][n] = ex;
            }
            const int f0 = sl.fmt[p][0], f1 = kDown ? f0 : sl.fmt[p][1];
            const int ks = (f0 == kQ80 || f1 == kQ80) ? 128 : 256;
            const GStage G = gstage(f0, f1, kTens, ks);
            if (G.total > kGPkBytes) {   // only the four formats above come here
                if (lane == 0) { fail(); s_unit[us].u = -1; mbar_arrive(uf + 8 * us); }
                break;
            }
            if (lane == 0) {
                GUnit g;
                g.u = u; g.p = p; g.mt = mt; g.N = N; g.Npad = (N + 15) & ~15; g.ks = ks; g.r0 = sl.first[p] + n0;
                s_unit[us] = g;
            }
            __syncwarp();
            if (lane == 0) mbar_arrive(uf + 8 * us);
            // this lane's copy: tensor z, plane pl, tile tl (lane = 16 z + 4 pl + tl)
            // (the per-lane choices are unrolled selects, so nothing is indexed at run time)
            const int z = lane >> 4, pl = (lane >> 2) & 3, tl = lane & 3;
            const int fz = z == 0 ? f0 : f1;
            const uint8_t* src0 = nullptr;
            int64_t sstep = 0;
            uint32_t bytes = 0, doff = 0;
#pragma unroll
            for (int zz = 0; zz < kTens; ++zz) {
                const int fm = zz == 0 ? f0 : f1;
                const PlaneBytes pb = plane_bytes(fm);
                const TensorLayout L = tensor_layout(fm, kDown ? d.H : d.I, K);
#pragma unroll
                for (int pp = 0; pp < 4; ++pp) {
                    if (zz == z && pp == pl && pp < pb.n) {
                        src0 = tab.p[sl.e[p]][zz == 0 ? (kDown ? 2 : 0) : 1] + L.plane[pp] +
                               unit_offset(L.blocks_per_row, pb.b[pp], (int64_t)mt * kMT + 32 * tl, 0, 0);
                        bytes = (uint32_t)G.tile[zz][pp];
                        doff = (uint32_t)(G.off[zz][pp] + tl * G.tile[zz][pp]);
                        sstep = (int64_t)32 * pb.b[pp];   // bytes per block of one tile
                    }
                }
            }
            const bool mine = bytes != 0;
            const int cps = ks / kKC;
            const int nst = (nC + cps - 1) / cps;   // a last K-quant superblock may hold 128 columns only
            bool bad = false;
            for (int st = 0; st < nst; ++st, ++pq) {
                const int ps = pq % kGPk;
                if (pq >= kGPk && !mbar_wait(pke + 8 * ps, ((pq - kGPk) / kGPk) & 1)) { bad = true; break; }
                if (failed()) { bad = true; break; }
                if (lane == 0) g_arrive_tx(pkf + 8 * ps, (uint32_t)G.total);
                __syncwarp();
                if (mine) {
                    const int64_t blk = fz == kQ80 ? (int64_t)st * (ks / 32) : (int64_t)st * ks / 256;
                    g_bulk(pk0 + ps * kGPkBytes + doff, src0 + blk * sstep, bytes, pkf + 8 * ps, pol);
                }
            }
            if (bad) { if (lane == 0) fail(); break; }
        }
        // the stages still in flight land before the CTA exits
        for (int q = max(0, pq - kGPk); q < pq; ++q) (void)mbar_wait(pkf + 8 * (q % kGPk), (q / kGPk) & 1);
    } else if (warp == kWarpB) {
        // ---- activations: the chunk's rows of the unit's tile, eight bulk copies
        // (one per 8-column piece) into the operand slot; the MMA may read rows
        // N .. Npad - 1 of an earlier chunk: they only reach accumulator
        // columns the epilogue never reads
        const uint8_t* src = kDown ? reinterpret_cast<const uint8_t*>(A.h16) : A.xp;
        int gq = 0;
        for (int ui = 0;; ++ui) {
            const int us = ui & 1;
            if (!mbar_wait(uf + 8 * us, (ui >> 1) & 1)) { if (lane == 0) fail(); break; }
            const GUnit U = s_unit[us];
            if (U.u < 0) break;
            bool bad = false;
            for (int c = 0; c < nC; ++c, ++gq) {
                const int s = gq % kGOps;
                if (gq >= kGOps && !mbar_wait(ope + 8 * s, ((gq - kGOps) / kGOps) & 1)) { bad = true; break; }
                if (failed()) { bad = true; break; }
                if (lane == 0) g_arrive_tx(opf + 8 * s, (uint32_t)(U.N * 128));
                __syncwarp();
                if (lane < 8)
                    asm volatile("cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];"
                                 ::"r"(ring + s * kGSlotBytes + kBOfs + lane * kGNT * 16),
                                   "l"(src + perm_piece(U.r0, K, U.N, c * 8 + lane, 0)), "r"((uint32_t)(U.N * 16)),
                                   "r"(opf + 8 * s) : "memory");
            }
            if (bad) { if (lane == 0) fail(); break; }
            __syncwarp();
            if (lane == 0) mbar_arrive(ue + 8 * us);
        }
    } else if (warp == kWarpM) {
        // ---- MMA issue.  The operand descriptors of both slots are built once:
        // a 16-column step of K moves an A operand by 2 * kMT * 16 bytes and B
        // by 2 * kGNT * 16 bytes, i.e. the descriptors' start-address field
        // (bytes / 16) by 256 and 512.
        uint64_t dA[kGOpsMax][2], dB[kGOpsMax];
#pragma unroll
        for (int sl2 = 0; sl2 < kGOpsMax; ++sl2) {
            const uint32_t sbase = ring + sl2 * kGSlotBytes;
            dA[sl2][0] = sdesc(sbase, kMT * 16, 128);
            dA[sl2][1] = sdesc(sbase + kABytes, kMT * 16, 128);
            dB[sl2] = sdesc(sbase + kBOfs, kGNT * 16, 128);
        }
        int mq = 0, last = -1;
        for (int ui = 0;; ++ui) {
            const int us = ui & 1;
            if (!mbar_wait(uf + 8 * us, (ui >> 1) & 1)) { if (lane == 0) fail(); break; }
            const GUnit U = s_unit[us];
            if (U.u < 0) break;
            bool bad = false;
            for (int c = 0; c < nC; ++c, ++mq) {
                const int s = mq % kGOps;
                if (!mbar_wait(opf + 8 * s, (mq / kGOps) & 1)) { bad = true; break; }
                if (lane == 0) {
                    // (the workers fenced their operand stores; the activations came by bulk copy)
                    asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
                    const uint32_t idesc = idesc_f16(kMT, U.Npad);
                    const uint64_t a0 = s == 0 ? dA[0][0] : s == 1 ? dA[1][0] : dA[2][0];
                    const uint64_t a1 = s == 0 ? dA[0][1] : s == 1 ? dA[1][1] : dA[2][1];
                    const uint64_t b0 = s == 0 ? dB[0] : s == 1 ? dB[1] : dB[2];
#pragma unroll
                    for (int kk = 0; kk < kKC / 16; ++kk) {
                        const uint32_t acc = (c > 0 || kk > 0) ? 1u : 0u;
                        mma_f16(tbase, a0 + 256u * kk, b0 + 512u * kk, idesc, acc);
                        if (!kDown) mma_f16(tbase + kGNT, a1 + 256u * kk, b0 + 512u * kk, idesc, acc);
                    }
                    asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];"
                                 ::"r"(ope + 8 * s) : "memory");
                }
                __syncwarp();
                last = mq;
            }
            if (bad) { if (lane == 0) fail(); break; }
            __syncwarp();
            if (lane == 0) mbar_arrive(ue + 8 * us);
        }
        // tensor memory is released only after the MMAs issued here are done
        if (last >= 0) (void)mbar_wait(ope + 8 * (last % kGOps), (last / kGOps) & 1);
    } else {
        // ---- workers: decode and epilogue.  Gate/up: warps 0-7 decode the gate
        // tensor, 8-15 the up tensor, of every chunk; down: warps 0-7 the even
        // chunks, 8-15 the odd ones.  Warp w takes the weight rows of tile w % 4
        // and half (w / 4) % 2 of its chunks.
        constexpr int nG = kDown ? 2 : 1;          // chunk groups
        const int z = kDown ? 0 : (warp >> 3);
        const int gsel = kDown ? (warp >> 3) : 0;
        const int tl = warp & 3, hf = (warp >> 2) & 1;
        const int rr = 32 * tl + lane;
        uint4* const sv4 = reinterpret_cast<uint4*>(smem);
        int gbase = 0, pbase = 0;   // chunks and packed stages of the earlier units
        for (int ui = 0;; ++ui) {
            const int us = ui & 1;
            if (!mbar_wait(uf + 8 * us, (ui >> 1) & 1)) { if (lane == 0) fail(); break; }
            const GUnit U = s_unit[us];
            if (U.u < 0) break;
            const int f0 = sl.fmt[U.p][0], f1 = kDown ? f0 : sl.fmt[U.p][1];
            const int fz = z ? f1 : f0;
            const GStage G = gstage(f0, f1, kTens, U.ks);
            uint32_t rec[4];   // this thread's records in stage 0 (stage s at + s * kGPkBytes)
#pragma unroll
            for (int pl = 0; pl < 4; ++pl)
                rec[pl] = pk0 + (uint32_t)((z ? G.off[1][pl] : G.off[0][pl]) + tl * (z ? G.tile[1][pl] : G.tile[0][pl]) +
                                           lane * (z ? G.ub[1][pl] : G.ub[0][pl]));
            const int cps = U.ks / kKC;
            bool bad = false;
            SBlk B;
            uint32_t so = 0;
            // one chunk: c its index in the unit, cc its 64-column quarter of the
            // superblock, lb its first Q8_0 block in the stage
            auto chunk = [&](int c, int cc, int lb, uint32_t so) -> bool {
                const int g = gbase + c, s = g % kGOps;
                if (g >= kGOps && !mbar_wait(ope + 8 * s, ((g - kGOps) / kGOps) & 1)) return false;
                if (failed()) return false;
                uint4* const dst = sv4 + (s * kGSlotBytes + z * kABytes) / 16 + rr;
                if (fz == kQ2K) {
                    dq_q2k(B, cc, hf, dst);
                } else if (fz == kQ3K) {
                    dq_q3k(B, cc, hf, dst);
                } else if (fz == kQ4K) {
                    dq_q4k(B, cc, hf, dst);
                } else {   // Q8_0: block lb + hf of the stage
                    const uint32_t cp = rec[1] + so + (lb + hf) * (32 * 32);
                    const uint4 w0 = g_lds128(cp), w1 = g_lds128(cp + 16);
                    const uint32_t w[8] = {w0.x, w0.y, w0.z, w0.w, w1.x, w1.y, w1.z, w1.w};
                    dq_q80(w, g_lds16(rec[0] + so + (lb + hf) * (32 * 2)), hf, dst);
                }
                // this thread's operand stores before the tensor cores read them
                asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
                mbar_arrive(opf + 8 * s);
                return true;
            };
            const int nst = (nC + cps - 1) / cps;
            for (int st = 0; st < nst && !bad; ++st) {
                const int q = pbase + st, ps = q % kGPk;
                if (!mbar_wait(pkf + 8 * ps, (q / kGPk) & 1)) { bad = true; break; }
                const uint32_t so = (uint32_t)(ps * kGPkBytes);
                if (fz != kQ80) {
                    const uint32_t r[4] = {rec[0] + so, rec[1] + so, rec[2] + so, rec[3] + so};
                    load_sblk_s(fz, r, hf, B);
                }
                if (cps == 4) {
                    // a whole superblock: the quarter index is a constant in each copy
#pragma unroll
                    for (int cl = 0; cl < 4; ++cl) {
                        const int c = 4 * st + cl;
                        if (c >= nC) break;
                        if (kDown && (cl & 1) != gsel) continue;
                        if (!chunk(c, cl, 0, so)) { bad = true; break; }
                    }
                } else {
                    // 128 columns (a Q8_0 tensor in the unit): one chunk per group
                    for (int cl = gsel; cl < 2; cl += nG) {
                        const int c = 2 * st + cl;
                        if (c >= nC) break;
                        if (!chunk(c, c & 3, 2 * cl, so)) { bad = true; break; }
                    }
                }
                if (bad) break;
                // every worker warp takes part in every stage: release it
                __syncwarp();
                if (lane == 0) mbar_arrive(pke + 8 * ps);
            }
            gbase += nC;
            pbase += (nC + cps - 1) / cps;
            if (bad) { if (lane == 0) fail(); break; }
            // the unit's MMAs are done once its last chunk's commit arrived.  The
            // slots' commits are awaited in chunk order: a phase-parity wait may
            // run at most one phase ahead of its barrier, and a warp that skipped
            // the other group's chunks has seen only every second completion
            for (int gg = max(0, gbase - kGOps); gg < gbase && !bad; ++gg)
                bad = !mbar_wait(ope + 8 * (gg % kGOps), (gg / kGOps) & 1);
            if (bad) { if (lane == 0) fail(); break; }
            asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
            // epilogue: TMEM lane 32 (w % 4) + lane = weight row; the worker
            // warps of a lane quarter take every (kW / 4)-th group of 8 columns
            const int row = U.mt * kMT + 32 * tl + lane;
            bool over = false;
            for (int n = 8 * (warp >> 2); n < U.Npad; n += 2 * kW) {
                uint32_t g8[8], u8[8];
                const uint32_t ta = tbase + ((uint32_t)(32 * tl) << 16) + (uint32_t)n;
                asm volatile("tcgen05.ld.sync.aligned.32x32b.x8.b32 {%0,%1,%2,%3,%4,%5,%6,%7}, [%8];"
                             : "=r"(g8[0]), "=r"(g8[1]), "=r"(g8[2]), "=r"(g8[3]), "=r"(g8[4]), "=r"(g8[5]),
                               "=r"(g8[6]), "=r"(g8[7]) : "r"(ta));
                if (!kDown)
                    asm volatile("tcgen05.ld.sync.aligned.32x32b.x8.b32 {%0,%1,%2,%3,%4,%5,%6,%7}, [%8];"
                                 : "=r"(u8[0]), "=r"(u8[1]), "=r"(u8[2]), "=r"(u8[3]), "=r"(u8[4]), "=r"(u8[5]),
                                   "=r"(u8[6]), "=r"(u8[7]) : "r"(ta + kGNT));
                asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
#pragma unroll
                for (int j = 0; j < 8; ++j) {
                    const int nn = n + j;
                    if (nn >= U.N) break;
                    const int a = s_asg[us][nn], ex = s_ex[us][nn];
                    if (kDown) {
                        A.pdn[(size_t)a * d.H + row] = ldexpf(__uint_as_float(g8[j]), 2 * ex);
                    } else {
                        const float gv = ldexpf(__uint_as_float(g8[j]), ex), uv = ldexpf(__uint_as_float(u8[j]), ex);
                        const float hs = ldexpf(silu(gv) * uv * s_w[us][nn], -2 * ex);
                        over |= !(fabsf(hs) <= 65504.0f);
                        // h in the down GEMM's activation layout (slot position U.r0 + nn)
                        *reinterpret_cast<__half*>(reinterpret_cast<uint8_t*>(A.h16) +
                                                   perm_piece(U.r0, d.I, U.N, row >> 3, nn) + (row & 7) * 2) =
                            __float2half_rn(hs);
                    }
                }
            }
            if (over) atomicOr(A.err, kErrRange);
            // the accumulators are read: the next unit's MMAs wait for this
            // thread's arrival on their operand slot
            asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
            __syncwarp();
            if (lane == 0) mbar_arrive(ue + 8 * us);
        }
    }
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
    cudaFuncSetAttribute(gemm_ws_kernel<false>, cudaFuncAttributeMaxDynamicSharedMemorySize, g_smem(false));
    cudaFuncSetAttribute(gemm_ws_kernel<true>, cudaFuncAttributeMaxDynamicSharedMemorySize, g_smem(true));
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
    A.xp = reinterpret_cast<uint8_t*>(w.pdn);   // dead until the down GEMM writes its partial rows
    if (!rare) {
        prof_begin("xperm", s);
        const cudaError_t ex = launch_pdl(xperm_kernel, dim3(4 * g_psms), dim3(kXpWarps * 32), 0, s,
                                          static_cast<const __half*>(w.x16), static_cast<const int32_t*>(w.offsets),
                                          static_cast<const int32_t*>(w.perm), static_cast<const int32_t*>(w.active),
                                          d, A.xp);
        prof_end(s);
        if (ex != cudaSuccess) return ex;
    }
    prof_begin("gateup_tc", s);
    cudaError_t err = rare ? launch_pdl(prefill_kernel<false, true>, dim3(g_psms), dim3(prefill_threads(false)), smem,
                                        s, tab, A)
                           : launch_pdl(gemm_ws_kernel<false>, dim3(g_psms), dim3(g_threads(false)), g_smem(false), s, tab, A);
    prof_end(s);
    if (err != cudaSuccess) return err;
    prof_begin("down_tc", s);
    err = rare ? launch_pdl(prefill_kernel<true, true>, dim3(g_psms), dim3(prefill_threads(true)), smem, s, tab, A)
               : launch_pdl(gemm_ws_kernel<true>, dim3(g_psms), dim3(g_threads(true)), g_smem(true), s, tab, A);
    prof_end(s);
    if (err != cudaSuccess) return err;
    return launch_combine(d, w.pdn, out, s);
}

}  // namespace mq
