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
// Work is cut into items (32 rows x 16 superblocks of one tensor of one
// expert x up to 4 tokens) taken from a global counter by one persistent CTA
// per SM.  The packed layout keeps any superblock range of a 32-row tile
// contiguous in every plane, so a producer warp streams each item through a
// 5-stage shared-memory ring with 1D bulk (TMA) copies that complete on
// mbarriers; 8 consumer warps (2 row tiles x 4 superblocks per stage) run
// the tensor-core math.  Item partial sums go to scratch; the last CTA to
// finish a row block combines them in a fixed order (SwiGLU for gate/up,
// routed + shared sum for down), so the results are deterministic.  Every
// wait on an mbarrier is bounded (about 1 s) and reports to an error word.
#include <cuda_fp16.h>

#include "mq_actprep.cuh"
#include "mq_internal.h"

namespace mq {
namespace {

constexpr unsigned kFull = 0xffffffffu;

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

// ---------------------------------------------------------------------------
// bulk-copy pipeline primitives (TMA 1D copies completing on mbarriers)
// ---------------------------------------------------------------------------
__device__ __forceinline__ void mbar_init(uint32_t bar, uint32_t count) {
    asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(bar), "r"(count) : "memory");
}
__device__ __forceinline__ void mbar_arrive(uint32_t bar) {
    asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(bar) : "memory");
}
__device__ __forceinline__ void mbar_arrive_tx(uint32_t bar, uint32_t bytes) {
    asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(bar), "r"(bytes) : "memory");
}
__device__ __forceinline__ bool mbar_try(uint32_t bar, uint32_t parity) {
    uint32_t ok;
    asm volatile(
        "{\n\t.reg .pred p;\n\tmbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\tselp.u32 %0, 1, 0, p;\n\t}"
        : "=r"(ok) : "r"(bar), "r"(parity) : "memory");
    return ok != 0;
}
__device__ __forceinline__ uint64_t global_ns() {
    uint64_t t;
    asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
    return t;
}
// Bounded wait: gives up after ~1 s, records `code` in the error word.
__device__ __forceinline__ bool mbar_wait(uint32_t bar, uint32_t parity, uint32_t* err, uint32_t code) {
    if (mbar_try(bar, parity)) return true;
    const uint64_t t0 = global_ns();
    for (;;) {
        if (mbar_try(bar, parity)) return true;
        if (global_ns() - t0 > 1000000000ull) { atomicOr(err, code); return false; }
    }
}
__device__ __forceinline__ void bulk_copy(uint32_t dst, const void* src, uint32_t bytes, uint32_t bar) {
    asm volatile("cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];"
                 ::"r"(dst), "l"(src), "r"(bytes), "r"(bar) : "memory");
}
__device__ __forceinline__ void consumer_sync() { asm volatile("bar.sync 1, %0;" ::"n"(512) : "memory"); }
__device__ __forceinline__ uint4 lds128(uint32_t a) {
    uint4 v;
    asm volatile("ld.shared.v4.u32 {%0,%1,%2,%3}, [%4];" : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w) : "r"(a));
    return v;
}
__device__ __forceinline__ uint2 lds64(uint32_t a) {
    uint2 v;
    asm volatile("ld.shared.v2.u32 {%0,%1}, [%2];" : "=r"(v.x), "=r"(v.y) : "r"(a));
    return v;
}
__device__ __forceinline__ uint32_t lds32(uint32_t a) {
    uint32_t v;
    asm volatile("ld.shared.u32 %0, [%1];" : "=r"(v) : "r"(a));
    return v;
}
__device__ __forceinline__ uint32_t lds16(uint32_t a) {
    unsigned short v;
    asm volatile("ld.shared.u16 %0, [%1];" : "=h"(v) : "r"(a));
    return v;
}
__device__ __forceinline__ uint32_t lds8(uint32_t a) {
    uint32_t v;
    asm volatile("ld.shared.u8 %0, [%1];" : "=r"(v) : "r"(a));
    return v;
}
__device__ __forceinline__ float ldsf(uint32_t a) { return __uint_as_float(lds32(a)); }

constexpr int kConsumers = 16;                      // consumer warps (the last also produces)
constexpr int kThreads = kConsumers * 32;
constexpr int kProducerWarp = kConsumers - 1;
constexpr int kNST = 4;                             // ring stages
constexpr int kStageBytes = 48 * 1024;
constexpr int kStageSb = 8;                         // superblocks per stage (Q8_0: 4), fewer if over budget
constexpr int kMaxCachedAssign = 2048;              // routed assignments cached in smem
constexpr uint32_t kErrFull = 1u, kErrEmpty = 2u;

struct DecodeArgs {
    Dims d;
    int nsbx, nsbi;          // superblocks along hidden / inter
    const __half* xq; const float* xs;   // prepared tokens
    __half* hq; float* hs;               // prepared SwiGLU outputs (per assignment)
    const int32_t* offsets; const int32_t* perm; const int32_t* active; const float* wts;
    const Plan* plan;
    float* pdn;              // [A][H]
    uint32_t* next;          // [2] item counters
    uint32_t* err;
    float* out;
};

// stage header written by the producer (one per ring slot)
struct Hdr {
    int32_t item, j, nst, s0, ks, kl;     // kl: superblocks the stage layout is sized for
    int32_t fmt, e, tensor, rb, tg, ntok, shared;
    int32_t vec[kDecodeTok], asg[kDecodeTok];
    int32_t woff[4];         // weight plane regions in the stage
    int32_t tok0, tstride;   // token regions
};

struct TokLay { int x, x1, sig, o, s, stride; };
__device__ __forceinline__ TokLay tok_lay(int fmt, int ks) {
    TokLay t;
    const bool wide = fmt == kQ4K || fmt == kQ80;
    int at = 0;
    t.x = at; at += ks * 512;
    t.x1 = at; if (fmt == kQ3K) at += ks * 512;
    t.sig = at; at += ks * 32;
    const int no = wide ? 8 : 16;
    t.o = at; at += ks * no * 4;
    t.s = at; if (fmt == kQ2K || fmt == kQ4K) at += ks * no * 4;
    t.stride = (at + 127) & ~127;
    return t;
}

__device__ __forceinline__ int weight_stage_bytes(int fmt, int ks) {
    const PlaneBytes pb = plane_bytes(fmt);
    const int nblk = fmt == kQ80 ? 8 * ks : ks;
    int at = 0;
    for (int p = 0; p < pb.n; ++p) at += (32 * nblk * pb.b[p] + 127) & ~127;
    return at;
}
// superblocks per stage for a format and token count (fits kStageBytes)
__device__ __forceinline__ int stage_sb(int fmt, int ntok) {
    int ks = fmt == kQ80 ? kStageSb / 2 : kStageSb;
    while (ks > 1 && weight_stage_bytes(fmt, ks) + ntok * tok_lay(fmt, ks).stride > kStageBytes) --ks;
    return ks;
}

// per-CTA cache of the routing result (slot -> expert, first entry, tokens)
struct SlotCache {
    int32_t e[kMaxExperts + 1], first[kMaxExperts + 1], ntot[kMaxExperts + 1];
    int32_t pre[kMaxExperts + 2];
};

struct ItemDesc {            // decoded item (producer side)
    int e, rb, tg, ntok, shared, nst0, nst;
    int vec[kDecodeTok], asg[kDecodeTok];
};

template <bool kDown>
__device__ __forceinline__ void decode_item(const DecodeArgs& A, const SlotCache& sc, const int32_t* s_perm, int n_slots,
                                            int id, int& cursor, const ExpertTab& tab, ItemDesc& it) {
    while (cursor + 1 < n_slots && sc.pre[cursor + 1] <= id) ++cursor;
    const int p = cursor;
    int local = id - sc.pre[p];
    const Dims& d = A.d;
    const int nrb = (kDown ? d.H : d.I) / 32;
    it.rb = local % nrb;
    it.tg = local / nrb;
    it.e = sc.e[p];
    it.shared = p < d.has_shared;
    it.ntok = min(kDecodeTok, sc.ntot[p] - it.tg * kDecodeTok);
    for (int j = 0; j < kDecodeTok; ++j) {
        int t = 0, a = 0;
        if (j < it.ntok) {
            const int q = it.tg * kDecodeTok + j;
            if (it.shared) { t = q; a = d.T * d.K + q; }
            else {
                const int idx = sc.first[p] + q;
                a = idx < kMaxCachedAssign ? s_perm[idx] : A.perm[idx];
                t = a / d.K;
            }
        }
        it.asg[j] = a;
        it.vec[j] = kDown ? a : t;
    }
    auto stages = [&](int fmt, int nsb) { const int per = stage_sb(fmt, it.ntok); return (nsb + per - 1) / per; };
    if (!kDown) {
        it.nst0 = stages(tab.fmt[it.e][0], A.nsbx);
        it.nst = it.nst0 + stages(tab.fmt[it.e][1], A.nsbx);
    } else {
        it.nst0 = stages(tab.fmt[it.e][2], A.nsbi);
        it.nst = it.nst0;
    }
}

// ---- consumer math: one warp = one 16-row tile x one superblock (Q8_0: half) ----
// x one token.  k-steps alternate between two accumulators (the two slot
// tiles of 16-wide sub-blocks, or even/odd steps of 32-wide ones) so
// consecutive MMAs are independent.  acc[h]: row g + 8h of the tile.
template <int FMT>
__device__ __forceinline__ void tile_token(const Hdr& h, uint32_t st, int jj, int half, int rt, int tk,
                                           float (&acc)[2]) {
    const int lane = threadIdx.x & 31, g = lane >> 2, t4 = lane & 3;
    constexpr bool kWide = FMT == kQ4K || FMT == kQ80;
    // ---- weights of rows (tile rt, g + 8 hl) for superblock jj of the stage
    uint32_t cw[2][8];
    uint32_t hw[2][2];
    uint32_t fld[2];
    float dd[2], dm[2];
    const int w0 = h.woff[0], w1 = h.woff[1], w2 = h.woff[2], w3 = h.woff[3];
#pragma unroll
    for (int hl = 0; hl < 2; ++hl) {
        const int r = 16 * rt + 8 * hl + g;
        fld[hl] = 0u; dm[hl] = 0.0f;
        if (FMT == kQ2K) {
            const uint4 c = lds128(st + w3 + (jj * 32 + r) * 64 + 16 * t4);
            cw[hl][0] = c.x; cw[hl][1] = c.y; cw[hl][2] = c.z; cw[hl][3] = c.w;
            fld[hl] = lds32(st + w2 + (jj * 32 + r) * 16 + 4 * t4);
            dd[hl] = h2f(lds16(st + w0 + (jj * 32 + r) * 2));
            dm[hl] = h2f(lds16(st + w1 + (jj * 32 + r) * 2));
        } else if (FMT == kQ3K) {
            const uint4 c = lds128(st + w2 + (jj * 32 + r) * 64 + 16 * t4);
            cw[hl][0] = c.x; cw[hl][1] = c.y; cw[hl][2] = c.z; cw[hl][3] = c.w;
            const uint2 hv = lds64(st + w3 + (jj * 32 + r) * 32 + 8 * t4);
            hw[hl][0] = hv.x; hw[hl][1] = hv.y;
            const uint32_t sp = st + w1 + (jj * 32 + r) * 12;
            fld[hl] = lds16(sp + 2 * t4) | (lds8(sp + 8 + t4) << 16);
            dd[hl] = h2f(lds16(st + w0 + (jj * 32 + r) * 2));
        } else if (FMT == kQ4K) {
            const uint4 c0 = lds128(st + w3 + ((jj * 2 + 0) * 32 + r) * 64 + 16 * t4);
            const uint4 c1 = lds128(st + w3 + ((jj * 2 + 1) * 32 + r) * 64 + 16 * t4);
            cw[hl][0] = c0.x; cw[hl][1] = c0.y; cw[hl][2] = c0.z; cw[hl][3] = c0.w;
            cw[hl][4] = c1.x; cw[hl][5] = c1.y; cw[hl][6] = c1.z; cw[hl][7] = c1.w;
            const uint32_t sp = st + w2 + (jj * 32 + r) * 12;
            fld[hl] = lds16(sp + 2 * t4) | (lds8(sp + 8 + t4) << 16);
            dd[hl] = h2f(lds16(st + w0 + (jj * 32 + r) * 2));
            dm[hl] = h2f(lds16(st + w1 + (jj * 32 + r) * 2));
        } else {  // Q8_0: blocks 8*jj + 4*half + (0..3)
#pragma unroll
            for (int q = 0; q < 4; ++q) {
                const uint2 v = lds64(st + w1 + ((8 * jj + 4 * half + q) * 32 + r) * 32 + 8 * t4);
                cw[hl][2 * q] = v.x; cw[hl][2 * q + 1] = v.y;
            }
            dd[hl] = h2f(lds16(st + w0 + ((8 * jj + 2 * t4) * 32 + r) * 2));
            dm[hl] = h2f(lds16(st + w0 + ((8 * jj + 2 * t4 + 1) * 32 + r) * 2));
        }
    }
    const TokLay tl = tok_lay(FMT, h.kl);
    const uint32_t tb = st + h.tok0 + tk * h.tstride;
    const uint4 X = lds128(tb + tl.x + jj * 512 + (g * 4 + t4) * 16);
    uint4 X1 = make_uint4(0, 0, 0, 0);
    if (FMT == kQ3K) X1 = lds128(tb + tl.x1 + jj * 512 + (g * 4 + t4) * 16);
    float D[2][4] = {{0.f, 0.f, 0.f, 0.f}, {0.f, 0.f, 0.f, 0.f}};
#pragma unroll
    for (int ii = 0; ii < (FMT == kQ80 ? 8 : 16); ++ii) {
        // 16-wide formats: i = 0, 8, 1, 9, ...; wide formats: in order (parity alternates)
        const int i = FMT == kQ80 ? 8 * half + ii : (kWide ? ii : ((ii >> 1) + 8 * (ii & 1)));
        const int owner = kWide ? (i >> 1) : (i & 7);
        const int sel = kWide ? (i & 1) : (i >> 3);
        const int acc_id = kWide ? (i & 1) : (i >> 3);
        // slot mask: only lanes of group `owner` supply the activations
        const uint32_t mk = g == owner ? 0x3C003C00u : 0u;
        uint32_t a[4];
        if (FMT == kQ2K || FMT == kQ3K) {
#pragma unroll
            for (int hl = 0; hl < 2; ++hl) {
                const uint32_t w = cw[hl][i >> 2], w10 = w >> 10;
                switch (i & 3) {
                case 0: a[hl] = ext2<0>(w, w10); a[2 + hl] = ext2<1>(w, w10); break;
                case 1: a[hl] = ext2<2>(w, w10); a[2 + hl] = ext2<3>(w, w10); break;
                case 2: a[hl] = ext2<4>(w, w10); a[2 + hl] = ext2<5>(w, w10); break;
                default: a[hl] = ext2<6>(w, w10); a[2 + hl] = ext2<7>(w, w10); break;
                }
            }
        } else if (FMT == kQ4K) {
#pragma unroll
            for (int hl = 0; hl < 2; ++hl) {
                const uint32_t w = cw[hl][4 * (i >> 3) + ((i & 7) >> 1)];
                const uint32_t ws = (i & 1) ? (w >> 8) : w;
                a[hl] = lop3_and_or(ws, 0x000F000Fu, 0x64006400u);
                a[2 + hl] = lop3_and_or(ws, 0x00F000F0u, 0x64006400u);
            }
        } else {
#pragma unroll
            for (int hl = 0; hl < 2; ++hl) {
                const uint32_t w = cw[hl][2 * ((i >> 1) - 4 * half) + (i & 1)];
                a[hl] = lop3_q8(w);
                a[2 + hl] = lop3_q8(w >> 8);
            }
        }
        const uint32_t b0 = hmul2u(sel ? X.z : X.x, mk);
        const uint32_t b1 = hmul2u(sel ? X.w : X.y, mk);
        mma16816(D[acc_id], a[0], a[1], a[2], a[3], b0, b1);
        if (FMT == kQ3K) {
            uint32_t ah[4];
#pragma unroll
            for (int hl = 0; hl < 2; ++hl) {
                const uint32_t w = hw[hl][i >> 3], w10 = w >> 10;
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
            const uint32_t c0 = hmul2u(sel ? X1.z : X1.x, mk);
            const uint32_t c1 = hmul2u(sel ? X1.w : X1.y, mk);
            mma16816(D[acc_id], ah[0], ah[1], ah[2], ah[3], c0, c1);
        }
    }
    // ---- epilogue: sub-block scales / mins in fp32
    if (FMT == kQ2K || FMT == kQ3K) {
        const uint4 Ou = lds128(tb + tl.o + jj * 64 + t4 * 16);
        const float Ov[4] = {__uint_as_float(Ou.x), __uint_as_float(Ou.y), __uint_as_float(Ou.z), __uint_as_float(Ou.w)};
        float Sv[4] = {0.f, 0.f, 0.f, 0.f};
        if (FMT == kQ2K) {
            const uint4 Su = lds128(tb + tl.s + jj * 64 + t4 * 16);
            Sv[0] = __uint_as_float(Su.x); Sv[1] = __uint_as_float(Su.y);
            Sv[2] = __uint_as_float(Su.z); Sv[3] = __uint_as_float(Su.w);
        }
        const float sg0 = ldsf(tb + tl.sig + (8 * jj + t4) * 4), sg1 = ldsf(tb + tl.sig + (8 * jj + 4 + t4) * 4);
#pragma unroll
        for (int hl = 0; hl < 2; ++hl) {
            float a_sc = 0.0f, a_m = 0.0f;
#pragma unroll
            for (int v = 0; v < 4; ++v) {   // v = 2*tile + e
                const float P = fmaf(D[v >> 1][2 * hl + (v & 1)], (v >> 1) ? sg1 : sg0, -Ov[v]);
                if (FMT == kQ2K) {
                    const uint32_t byte = (fld[hl] >> (8 * v)) & 0xffu;
                    a_sc = fmaf((float)(byte & 15u), P, a_sc);
                    a_m = fmaf((float)(byte >> 4), Sv[v], a_m);
                } else {
                    const uint32_t f = fld[hl];
                    const int sfield = (int)((f >> (4 * v)) & 15u) | (int)(((f >> (16 + 2 * v)) & 3u) << 4);
                    a_sc = fmaf((float)(sfield - 32), P, a_sc);
                }
            }
            float r = dd[hl] * a_sc;
            if (FMT == kQ2K) r = fmaf(-dm[hl], a_m, r);
            acc[hl] += r;
        }
    } else {
        const uint2 Ou = lds64(tb + tl.o + (8 * jj + 2 * t4) * 4);
        const uint2 Gu = lds64(tb + tl.sig + (8 * jj + 2 * t4) * 4);
        const float O0 = __uint_as_float(Ou.x), O1 = __uint_as_float(Ou.y);
        const float sg0 = __uint_as_float(Gu.x), sg1 = __uint_as_float(Gu.y);
        float S0 = 0.f, S1 = 0.f;
        if (FMT == kQ4K) {
            const uint2 Su = lds64(tb + tl.s + (8 * jj + 2 * t4) * 4);
            S0 = __uint_as_float(Su.x); S1 = __uint_as_float(Su.y);
        }
        // Q8_0: this half holds blocks 4*half..4*half+3; lane t4 owns blocks 2*t4, 2*t4+1
        if (FMT == kQ4K || (t4 >> 1) == half) {
#pragma unroll
            for (int hl = 0; hl < 2; ++hl) {
                const float D0 = D[0][2 * hl] + D[1][2 * hl];
                const float D1 = D[0][2 * hl + 1] + D[1][2 * hl + 1];
                const float P0 = fmaf(D0, sg0, -O0), P1 = fmaf(D1, sg1, -O1);
                if (FMT == kQ4K) {
                    const uint32_t f = fld[hl];
                    const int hi = (int)(f >> 16);
                    const float sc0 = (float)((f & 15u) | ((hi & 3) << 4));
                    const float m0 = (float)(((f >> 4) & 15u) | (((hi >> 2) & 3) << 4));
                    const float sc1 = (float)(((f >> 8) & 15u) | (((hi >> 4) & 3) << 4));
                    const float m1 = (float)(((f >> 12) & 15u) | (((hi >> 6) & 3) << 4));
                    const float a_sc = fmaf(sc1, P1, sc0 * P0);
                    const float a_m = fmaf(m1, S1, m0 * S0);
                    acc[hl] += fmaf(dd[hl], a_sc, -dm[hl] * a_m);
                } else {
                    acc[hl] += fmaf(dd[hl], P0, dm[hl] * P1);
                }
            }
        }
    }
}

template <bool kDown>
__global__ void __launch_bounds__(kThreads, 1) ffn_kernel(const __grid_constant__ ExpertTab tab,
                                                          const __grid_constant__ DecodeArgs A) {
    extern __shared__ __align__(128) uint8_t smem[];
    __shared__ SlotCache sc;
    __shared__ int32_t s_perm[kMaxCachedAssign];
    __shared__ __align__(8) uint64_t bars[2 * kNST];
    __shared__ Hdr hdr[kNST];
    __shared__ float red[2][kConsumers][2][kDecodeTok][16];   // double-buffered by item parity
    __shared__ int s_posted[kNST];   // last stage index posted to each ring slot
    const Dims& d = A.d;
    const int n_slots = A.plan->n_slots;
    for (int i = threadIdx.x; i <= n_slots; i += blockDim.x) {
        sc.pre[i] = kDown ? A.plan->pre_dn[i] : A.plan->pre_gu[i];
        if (i < n_slots) {
            if (i < d.has_shared) { sc.e[i] = d.E; sc.first[i] = 0; sc.ntot[i] = d.T; }
            else {
                const int e = A.active[1 + i - d.has_shared];
                sc.e[i] = e; sc.first[i] = A.offsets[e]; sc.ntot[i] = A.offsets[e + 1] - A.offsets[e];
            }
        }
    }
    const int n_routed = min(d.T * d.K, kMaxCachedAssign);
    for (int i = threadIdx.x; i < n_routed; i += blockDim.x) s_perm[i] = A.perm[i];
    const uint32_t bar0 = (uint32_t)__cvta_generic_to_shared(bars);
    if (threadIdx.x < kNST) s_posted[threadIdx.x] = -1;
    if (threadIdx.x == 0) {
        for (int s = 0; s < kNST; ++s) {
            mbar_init(bar0 + 8 * s, 1);                       // full[s]: producer arrival + tx bytes
            mbar_init(bar0 + 8 * (kNST + s), kConsumers);     // empty[s]: one arrival per consumer warp
        }
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    }
    __syncthreads();
    const int n_items = sc.pre[n_slots];
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const uint32_t ring = (uint32_t)__cvta_generic_to_shared(smem);
    const VecSrc vs = kDown ? VecSrc{A.hq, A.hs, (size_t)4 * A.nsbi * 256, (size_t)stat_off(A.nsbi).total, A.nsbi}
                            : VecSrc{A.xq, A.xs, (size_t)4 * A.nsbx * 256, (size_t)stat_off(A.nsbx).total, A.nsbx};

    // ====================== producer (run by warp 7) ========================
    // Per phase (one tensor of one item) every lane of warp 7 owns at most one
    // copy: lanes 0..3 a weight plane, lanes 4.. one piece of one token
    // (fragments, high-bit fragments, sigma, offsets, sums).  A stage then only
    // advances the source by the stage's first superblock.
    int p_cursor = 0, p_item = -1, p_j = 0, p_q = 0, p_nst = 0, p_nst0 = 0;
    int p_phase_j = 0, p_per = 1, p_nsb = vs.nsb, p_fmt = 0, p_tensor = 0;
    bool p_failed = false, p_done = false;
    const uint8_t* c_src = nullptr;       // this lane's copy: source at superblock 0
    uint32_t c_stride = 0, c_dst = 0;     // bytes per superblock, offset in the stage
    int h_woff0 = 0, h_woff1 = 0, h_woff2 = 0, h_woff3 = 0, h_tok0 = 0, h_tstride = 0;
    ItemDesc P;
    P.nst = 0; P.ntok = 0;
    const StatOff so = stat_off(vs.nsb);
    int next_id = 0;
    if (warp == kProducerWarp && lane == 0) next_id = (int)atomicAdd(&A.next[kDown ? 1 : 0], 1u);

#define MQ_PRODUCE_ONE()                                                                                   \
    do {                                                                                                   \
        if (p_done) break;                                                                                 \
        if (p_j == p_nst) {                                                                                \
            const int id = __shfl_sync(kFull, next_id, 0);                                                 \
            p_item = id < n_items ? id : -1;                                                               \
            if (p_item >= 0) {                                                                             \
                decode_item<kDown>(A, sc, s_perm, n_slots, p_item, p_cursor, tab, P);                     \
                if (lane == 0) next_id = (int)atomicAdd(&A.next[kDown ? 1 : 0], 1u);                       \
                p_nst = P.nst; p_nst0 = P.nst0;                                                            \
            }                                                                                              \
            p_j = 0;                                                                                       \
        }                                                                                                  \
        const int slot = p_q % kNST;                                                                       \
        const uint32_t full = bar0 + 8 * slot, empty = bar0 + 8 * (kNST + slot);                            \
        if (p_q >= kNST && !mbar_wait(empty, ((p_q / kNST) & 1) ^ 1, A.err, kErrEmpty)) {                \
            p_failed = true; p_done = true; break;                                                         \
        }                                                                                                  \
        if (p_item < 0) {                                                                                  \
            if (lane == 0) { hdr[slot].item = -1; s_posted[slot] = p_q; mbar_arrive(full); }              \
            p_done = true;                                                                                 \
            break;                                                                                         \
        }                                                                                                  \
        if (p_j == 0 || (!kDown && p_j == p_nst0)) {                                                       \
            /* new phase: tensor, format, stage geometry, this lane's copy */                             \
            p_tensor = kDown ? 2 : (p_j == 0 ? 0 : 1);                                                     \
            p_phase_j = p_j;                                                                               \
            p_fmt = tab.fmt[P.e][p_tensor];                                                                \
            p_per = stage_sb(p_fmt, P.ntok);                                                               \
            const TensorLayout L = tensor_layout(p_fmt, kDown ? d.H : d.I, kDown ? d.I : d.H);            \
            const PlaneBytes pb = plane_bytes(p_fmt);                                                      \
            const int bmul = p_fmt == kQ80 ? 8 : 1;                                                        \
            int at = 0, wo[4] = {0, 0, 0, 0};                                                              \
            _Pragma("unroll") for (int pl = 0; pl < 4; ++pl) {                                             \
                wo[pl] = at;                                                                               \
                if (pl < pb.n) at += (32 * bmul * p_per * pb.b[pl] + 127) & ~127;                          \
            }                                                                                              \
            h_woff0 = wo[0]; h_woff1 = wo[1]; h_woff2 = wo[2]; h_woff3 = wo[3];                            \
            const TokLay tl = tok_lay(p_fmt, p_per);                                                       \
            h_tok0 = at; h_tstride = tl.stride;                                                            \
            c_src = nullptr; c_stride = 0; c_dst = 0;                                                      \
            const uint8_t* tbase = tab.p[P.e][p_tensor];                                                   \
            _Pragma("unroll") for (int pl = 0; pl < 4; ++pl)                                               \
                if (lane == pl && pl < pb.n) {                                                             \
                    c_src = tbase + L.plane[pl] + (int64_t)P.rb * L.blocks_per_row * 32 * pb.b[pl];        \
                    c_stride = 32 * bmul * pb.b[pl];                                                       \
                    c_dst = wo[pl];                                                                        \
                }                                                                                          \
            if (lane >= 4 && lane < 4 + 5 * P.ntok) {                                                      \
                const int tk = (lane - 4) / 5, piece = (lane - 4) % 5;                                     \
                int v = P.vec[0];                                                                          \
                _Pragma("unroll") for (int t2 = 1; t2 < kDecodeTok; ++t2) if (tk == t2) v = P.vec[t2];     \
                const uint8_t* qv = reinterpret_cast<const uint8_t*>(vs.q + (size_t)v * vs.q_stride);      \
                const uint8_t* sv = reinterpret_cast<const uint8_t*>(vs.st + (size_t)v * vs.st_stride);    \
                const int fam = p_fmt == kQ2K || p_fmt == kQ3K ? kF2 : p_fmt == kQ4K ? kF4 : kF8;          \
                const bool wide = p_fmt == kQ4K || p_fmt == kQ80;                                          \
                const uint32_t tb = h_tok0 + tk * tl.stride;                                               \
                if (piece == 0) { c_src = qv + (size_t)fam * vs.nsb * 512; c_stride = 512; c_dst = tb + tl.x; } \
                if (piece == 1 && p_fmt == kQ3K) {                                                         \
                    c_src = qv + (size_t)kF1 * vs.nsb * 512; c_stride = 512; c_dst = tb + tl.x1;           \
                }                                                                                          \
                if (piece == 2) { c_src = sv + 4 * so.sig; c_stride = 32; c_dst = tb + tl.sig; }            \
                if (piece == 3) {                                                                          \
                    const int o = p_fmt == kQ2K ? so.os2 : p_fmt == kQ3K ? so.oq3 : p_fmt == kQ4K ? so.os4 : so.os8; \
                    c_src = sv + 4 * o; c_stride = wide ? 32 : 64; c_dst = tb + tl.o;                       \
                }                                                                                          \
                if (piece == 4 && (p_fmt == kQ2K || p_fmt == kQ4K)) {                                      \
                    c_src = sv + 4 * (p_fmt == kQ2K ? so.sxs16 : so.sxs32); c_stride = wide ? 32 : 64;     \
                    c_dst = tb + tl.s;                                                                     \
                }                                                                                          \
            }                                                                                              \
        }                                                                                                  \
        const int s0 = (p_j - p_phase_j) * p_per, ks = min(p_per, p_nsb - s0);                             \
        const uint32_t stage = ring + slot * kStageBytes;                                                  \
        const uint32_t bytes = c_src ? (uint32_t)ks * c_stride : 0u;                                       \
        uint32_t total = bytes;                                                                            \
        _Pragma("unroll") for (int off = 16; off >= 1; off >>= 1) total += __shfl_xor_sync(kFull, total, off); \
        if (lane == 0) {                                                                                   \
            Hdr& H = hdr[slot];                                                                            \
            H.item = p_item; H.j = p_j; H.nst = p_nst; H.s0 = s0; H.ks = ks; H.kl = p_per;                  \
            H.fmt = p_fmt; H.e = P.e; H.tensor = p_tensor; H.rb = P.rb; H.tg = P.tg; H.ntok = P.ntok;      \
            H.shared = P.shared;                                                                           \
            _Pragma("unroll") for (int t2 = 0; t2 < kDecodeTok; ++t2) { H.vec[t2] = P.vec[t2]; H.asg[t2] = P.asg[t2]; } \
            H.woff[0] = h_woff0; H.woff[1] = h_woff1; H.woff[2] = h_woff2; H.woff[3] = h_woff3;            \
            H.tok0 = h_tok0; H.tstride = h_tstride;                                                        \
            s_posted[slot] = p_q;                                                                          \
            mbar_arrive_tx(full, total);                                                                   \
        }                                                                                                  \
        __syncwarp();                                                                                      \
        if (bytes) bulk_copy(stage + c_dst, c_src + (size_t)s0 * c_stride, bytes, full);                   \
        ++p_j;                                                                                             \
        ++p_q;                                                                                             \
    } while (0)

    if (warp == kProducerWarp)
        for (int i = 0; i < kNST - 1; ++i) MQ_PRODUCE_ONE();

    // ============================ consumer warps =============================
    // warp w: row tile w & 1; superblock w >> 1 of the stage (Q8_0: superblock
    // w >> 2, half (w >> 1) & 1)
    const int rt = warp & 1;
    float acc[2][kDecodeTok][2];   // [0] gate (or down), [1] up; rows g, g+8 of the tile
    float cur[kDecodeTok][2];      // the tensor being streamed
#pragma unroll
    for (int tk = 0; tk < kDecodeTok; ++tk) {
        acc[0][tk][0] = acc[0][tk][1] = acc[1][tk][0] = acc[1][tk][1] = 0.0f;
        cur[tk][0] = cur[tk][1] = 0.0f;
    }
    int n_done = 0;   // items finished by this CTA (selects the reduction buffer and the owner warps)
    for (int q = 0;; ++q) {
        if (warp == kProducerWarp) MQ_PRODUCE_ONE();   // posts stage q + kNST - 1
        const int slot = q % kNST;
        if (!mbar_wait(bar0 + 8 * slot, (q / kNST) & 1, A.err, kErrFull)) { p_failed = true; break; }
        const Hdr& H = hdr[slot];
        if (H.item < 0) break;
        const uint32_t stage = ring + slot * kStageBytes;
        const bool q8 = H.fmt == kQ80;
        const int sbj = q8 ? (warp >> 2) : (warp >> 1), half = q8 ? ((warp >> 1) & 1) : 0;
        if (!kDown && H.tensor == 1 && H.s0 == 0) {
            // first stage of the up tensor: the gate sums are complete
#pragma unroll
            for (int tk = 0; tk < kDecodeTok; ++tk) {
                acc[0][tk][0] += cur[tk][0]; acc[0][tk][1] += cur[tk][1];
                cur[tk][0] = cur[tk][1] = 0.0f;
            }
        }
        if (sbj < H.ks) {
            const int ntok = H.ntok;
#pragma unroll
            for (int tk = 0; tk < kDecodeTok; ++tk) {
                if (tk >= ntok) break;
                switch (H.fmt) {
                case kQ2K: tile_token<kQ2K>(H, stage, sbj, half, rt, tk, cur[tk]); break;
                case kQ3K: tile_token<kQ3K>(H, stage, sbj, half, rt, tk, cur[tk]); break;
                case kQ4K: tile_token<kQ4K>(H, stage, sbj, half, rt, tk, cur[tk]); break;
                default: tile_token<kQ80>(H, stage, sbj, half, rt, tk, cur[tk]); break;
                }
            }
        }
        // fields needed after the slot is released to the producer
        const bool item_end = H.j == H.nst - 1;
        int e_rb = 0, e_ntok = 0, e_shared = 0, e_e = 0;
        int e_asg[kDecodeTok];
        if (item_end) {
            e_rb = H.rb; e_ntok = H.ntok; e_shared = H.shared; e_e = H.e;
#pragma unroll
            for (int tk = 0; tk < kDecodeTok; ++tk) e_asg[tk] = H.asg[tk];
        }
        __syncwarp();
        if (lane == 0) mbar_arrive(bar0 + 8 * (kNST + slot));
        if (!item_end) continue;

        // ---- item done: the streamed tensor's sums go to acc[1] (up) or acc[0]
        const int g = lane >> 2, t4 = lane & 3;
        const int buf = n_done & 1;
#pragma unroll
        for (int u = 0; u < (kDown ? 1 : 2); ++u)
#pragma unroll
            for (int tk = 0; tk < kDecodeTok; ++tk)
#pragma unroll
                for (int hl = 0; hl < 2; ++hl) {
                    float v = (u == (kDown ? 0 : 1)) ? acc[u][tk][hl] + cur[tk][hl] : acc[u][tk][hl];
                    v += __shfl_xor_sync(kFull, v, 1);
                    v += __shfl_xor_sync(kFull, v, 2);
                    if (t4 == 0) red[buf][warp][u][tk][8 * hl + g] = v;
                }
#pragma unroll
        for (int tk = 0; tk < kDecodeTok; ++tk) {
            acc[0][tk][0] = acc[0][tk][1] = acc[1][tk][0] = acc[1][tk][1] = 0.0f;
            cur[tk][0] = cur[tk][1] = 0.0f;
        }
        consumer_sync();
        // the finishing work of token tk goes to warp (n_done + tk) % kConsumers
        const int tk = (warp - n_done % kConsumers + kConsumers) % kConsumers;
        if (tk < e_ntok) {
            int a = e_asg[0];
#pragma unroll
            for (int t2 = 1; t2 < kDecodeTok; ++t2) if (tk == t2) a = e_asg[t2];
            // lane = row of the 32-row block: row tile lane/16, row lane%16
            const int ort = lane >> 4, rr = lane & 15;
            float v0 = 0.0f, v1 = 0.0f;
#pragma unroll
            for (int sb = 0; sb < kConsumers / 2; ++sb) {
                v0 += red[buf][2 * sb + ort][0][tk][rr];
                if (!kDown) v1 += red[buf][2 * sb + ort][1][tk][rr];
            }
            if (kDown) {
                A.pdn[(size_t)a * d.H + 32 * e_rb + lane] = v0;
            } else {
                // SwiGLU (routing weight folded in), then prepare h for the down projection
                const float w = e_shared ? 1.0f : A.wts[a];
                const float hv = v0 / (1.0f + expf(-v0)) * v1 * w;
                const int fam = families_of(tab.fmt[e_e][2]);
                __half* hq = A.hq + (size_t)a * 4 * A.nsbi * 256;
                float* hs = A.hs + (size_t)a * stat_off(A.nsbi).total;
                prep_block32(hv, e_rb, fam, hq, hs, A.nsbi);
                const int n_rb = d.I / 32;
                if (e_rb == n_rb - 1)
                    for (int jb = n_rb; jb < 8 * A.nsbi; ++jb) prep_block32(0.0f, jb, fam, hq, hs, A.nsbi);
            }
        }
        // no barrier here: the next item end writes the other reduction buffer,
        // and its barrier orders these reads before the buffer is reused
        ++n_done;
    }
#undef MQ_PRODUCE_ONE
    // After a wait ran out, wait (bounded) for the copies still in flight into
    // each slot before the CTA exits.  Normally every posted stage has been
    // consumed, so nothing is in flight.
    if (warp == kProducerWarp) {
        __syncwarp();
        if (p_failed && lane < kNST && s_posted[lane] >= 0)
            mbar_wait(bar0 + 8 * lane, (s_posted[lane] / kNST) & 1, A.err, kErrFull);
    }
}

// out[t] = sum of the token's routed expert outputs in slot order, then the
// shared expert (deterministic order; routing weights are folded into h)
__global__ void combine_kernel(Dims d, const float* __restrict__ pdn, float* __restrict__ out) {
    const int r = blockIdx.x * blockDim.x + threadIdx.x;
    if (r >= d.H) return;
    for (int t = blockIdx.y; t < d.T; t += gridDim.y) {
        float y = 0.0f;
        for (int j = 0; j < d.K; ++j) y += __ldg(pdn + (size_t)(t * d.K + j) * d.H + r);
        if (d.has_shared) y += __ldg(pdn + (size_t)(d.T * d.K + t) * d.H + r);
        out[(size_t)t * d.H + r] = y;
    }
}

int g_num_sms = 0;

}  // namespace

size_t decode_counter_bytes(const Dims& d) {
    (void)d;
    return 2 * 4;   // gate/up and down item counters
}

cudaError_t launch_decode_mma(const Dims& d, const ExpertTab& tab, const Work& w, float* out, cudaStream_t s) {
    if (d.T == 0) return cudaSuccess;
    const int smem = kNST * kStageBytes;
    if (g_num_sms == 0) {
        int dev = 0;
        cudaGetDevice(&dev);
        cudaDeviceGetAttribute(&g_num_sms, cudaDevAttrMultiProcessorCount, dev);
        if (g_num_sms <= 0) g_num_sms = 148;
        cudaFuncSetAttribute(ffn_kernel<false>, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
        cudaFuncSetAttribute(ffn_kernel<true>, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
    }
    DecodeArgs A;
    A.d = d;
    A.nsbx = (d.H + 255) / 256;
    A.nsbi = (d.I + 255) / 256;
    A.xq = w.xq; A.xs = w.xs; A.hq = w.hq; A.hs = w.hs;
    A.offsets = w.offsets; A.perm = w.perm; A.active = w.active; A.wts = w.wts;
    A.plan = w.plan;
    A.pdn = w.pdn;
    A.next = w.counters;
    A.err = w.err;
    A.out = out;
    prof_begin("gateup_mma", s);
    ffn_kernel<false><<<g_num_sms, kThreads, smem, s>>>(tab, A);
    prof_end(s);
    cudaError_t err = cudaGetLastError();
    if (err != cudaSuccess) return err;
    prof_begin("down_mma", s);
    ffn_kernel<true><<<g_num_sms, kThreads, smem, s>>>(tab, A);
    prof_end(s);
    err = cudaGetLastError();
    if (err != cudaSuccess) return err;
    prof_begin("combine", s);
    combine_kernel<<<dim3((d.H + 255) / 256, d.T < 8 ? d.T : 8), 256, 0, s>>>(d, w.pdn, out);
    prof_end(s);
    return cudaGetLastError();
}

}  // namespace mq
