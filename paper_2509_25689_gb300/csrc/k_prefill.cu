// Expert FFN for prefill-sized batches: a grouped GEMM per expert on the
// 5th-generation tensor cores (arXiv 2509.25689 Fig. 1 layer; expert tensors
// in their own k-quant style formats, Sec. 3.3).
//
// Work unit = (expert slot, 128 weight rows, up to 256 of the slot's tokens).
// The MMA is tcgen05.mma.cta_group::1.kind::f16 with M = 128 weight rows,
// N = the unit's tokens (rounded up to 16) and K in steps of 16, fp32
// accumulators in tensor memory (gate and up side by side for gate/up units).
// The weights are dequantized to fp16 in shared memory, 64 contraction
// columns (a chunk) at a time (fp16 keeps 11 significant bits of a decoded
// weight); operands sit in the canonical K-major layout without swizzle:
// 8 x 8 fp16 core matrices, 16 bytes per row, rows of a core matrix
// contiguous, core matrices 128 bytes apart along M/N and (rows x 16) bytes
// apart along K.
// Epilogue (tcgen05.ld, lane = weight row): gate/up -> h = silu(g) * u * w
// stored as fp16 in the down GEMM's activation layout; down -> one fp32
// partial output row block per assignment, summed in slot order by the
// combine kernel.  Range: token t enters as fp16(x * 2^-e_t), e_t = the
// exponent of its largest |x| (so any finite bf16 token fits), and h as
// fp16(h * 2^-2 e_t); the epilogues undo both scalings in fp32.  An h that
// would still overflow fp16 sets an error bit (MQ_EDEVICE from
// moe_quant_status) instead of passing an inf on, and so does a BF16 weight
// beyond the fp16 range.  Every mbarrier wait is bounded (about 1 s) and
// reports to the error word; tensor memory is released on every exit path.
#include <cuda_fp16.h>

#include <type_traits>

#include "mq_internal.h"

namespace mq {
namespace {

constexpr int kMT = 128;                       // weight rows per unit (MMA M)
constexpr int kKC = 64;                        // K per ring slot
constexpr int kABytes = kMT * kKC * 2;         // one weight chunk, 16 KB
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
__device__ __forceinline__ uint32_t h2u(__half2 h) { return *reinterpret_cast<uint32_t*>(&h); }
__device__ __forceinline__ __half2 u2h(uint32_t u) { return *reinterpret_cast<__half2*>(&u); }
// One superblock's packed fields of one weight row for this thread's half of
// each of its four 64-wide chunks (Q2_K, Q3_K, Q4_K): codes, scales and d /
// dmin, read from the staged records once per stage.
struct SBlk {
    uint4 cw[4];      // Q2_K / Q3_K low bits: words 4i..4i+3 for i = 2 hf, 2 hf + 1; Q4_K: the 4 chunks' 16 bytes
    uint2 hw[2];      // Q3_K high bits: words 2i, 2i+1
    uint32_t sc[4];   // scale record
    uint32_t dd;      // d | dmin << 16
};
__device__ __forceinline__ float silu(float v) { return v / (1.0f + expf(-v)); }

// ---------------------------------------------------------------------------
// The GEMM kernel is warp-specialised: each CTA runs four roles at once, so
// that the record loads, the weight decode, the activation copies and the
// MMAs of different chunks overlap instead of following one another:
//   - a producer warp claims the units, publishes each one (slot, rows,
//     tokens) in a two-deep unit ring and streams the unit's packed records
//     into a two-stage ring with bulk copies (one per tensor, plane and
//     32-row tile; a stage holds one superblock, 128 contraction columns
//     when a tensor is Q8_0 or Q6_K, 64 when one is BF16; a K-quant partner's
//     superblock record then comes again with every stage of its superblock);
//   - sixteen worker warps decode the records from shared memory into the
//     fp16 operand of each chunk (gate/up: eight warps per tensor, down:
//     eight per chunk parity) and, at the unit's end, run the epilogue out
//     of tensor memory; the gate/up epilogue writes h straight into the down
//     GEMM's activation layout;
//   - an activation warp moves the chunk's activation rows with one bulk
//     copy from the tile-ordered copy of the tokens (xperm_kernel) or of h;
//   - an MMA warp issues a chunk's MMAs once the workers and the activation
//     warp have filled its operand slot (a two-slot ring) and commits them
//     to the slot's empty barrier.
// Every wait is bounded and reports to the error word.
// 16 worker warps (gate/up: 8 per tensor; down: 8 per chunk parity), then
// the producer, activation and MMA warps
__host__ __device__ constexpr int g_workers(bool down) { return 16; }
__host__ __device__ constexpr int g_threads(bool down) { return (g_workers(down) + 3) * 32; }
#ifndef MQ_GNT
#define MQ_GNT 256
#endif
#ifndef MQ_GOPS_GU
#define MQ_GOPS_GU 2
#endif
#ifndef MQ_GOPS_DN
#define MQ_GOPS_DN 3
#endif
#ifndef MQ_GPK
#define MQ_GPK 2
#endif
constexpr int kGNT = MQ_GNT;                   // tokens per unit (MMA N up to 256)
// operand slots: gate/up two of A gate | A up | B (64 KB), down three of
// A | B (48 KB); a third gate/up slot fits only with 128-token units,
// measured slower on the Zipf prefill
__host__ __device__ constexpr int g_ops(bool down) { return down ? MQ_GOPS_DN : MQ_GOPS_GU; }
__host__ __device__ constexpr int g_bofs(bool down) { return down ? kABytes : 2 * kABytes; }
__host__ __device__ constexpr int g_slot(bool down) { return g_bofs(down) + kGNT * kKC * 2; }
constexpr int kGOpsMax = MQ_GOPS_GU > MQ_GOPS_DN ? MQ_GOPS_GU : MQ_GOPS_DN;
constexpr int kGPk = MQ_GPK;                   // packed-record stages
constexpr int kGPkBytes = 37376;               // Q6_K + Q6_K half superblock of 128 rows: 2 x 18,688
__host__ __device__ constexpr int g_smem(bool down) { return g_ops(down) * g_slot(down) + kGPk * kGPkBytes; }
// a unit's tokens are the MMA's N (at most 256) and its TMEM columns (a power
// of two); the dynamic shared memory leaves room for the kernel's static
// arrays (about 7 KB) within the 227 KB of a CTA
static_assert(kGNT >= 32 && kGNT <= 256 && (kGNT & (kGNT - 1)) == 0, "tokens per unit");
static_assert(kGOpsMax >= 2 && kGOpsMax <= 4 && kGPk >= 2, "ring depths");
static_assert(g_smem(false) <= 219 * 1024 && g_smem(true) <= 219 * 1024, "shared memory per CTA");

// Activation rows of the warp-specialised GEMM in the order its units read
// them: slot positions r (the permutation's order for the routed experts,
// T*K + t for the shared expert), cut into tiles of up to kGNT rows of one
// slot.  In a tile of N rows starting at position r0, the 16-byte piece p
// (columns 8p .. 8p+7) of row n sits (p * N + n) * 16 bytes after r0 * K * 2,
// so a 64-column chunk of a tile is one contiguous run of 8 x N x 16 bytes:
// one bulk copy into the canonical operand layout whose core matrices are
// N x 16 bytes apart along K.
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
        const int nb = block_len(f) == 32 ? ks / 32 : 1;
#pragma unroll
        for (int pl = 0; pl < 4; ++pl) {
            const bool on = z < ntens && pl < pb.n;
            G.off[z][pl] = at;
            // (Q6_K's low-nibble record: only the 64-byte unit of the stage's half)
            G.tile[z][pl] = on ? nb * 32 * (f == kQ6K && pl == 2 ? 64 : pb.b[pl]) : 0;
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
__device__ __forceinline__ uint4 pick4(const uint4 (&v)[4], int i) {
    const uint4 a = (i & 1) ? v[1] : v[0], b = (i & 1) ? v[3] : v[2];
    return (i & 2) ? b : a;
}

// ---- chunk decode: each thread turns 32 weights of its row into fp16 in
// the A operand.  Roundings: d * sc and dmin * m (exact products) are rounded
// to fp16 once, then one fused multiply-add per weight pair.  A code field at
// bit s <= 8 of each 16-bit half, OR-ed into the fp16 pair 2^(10 - s), reads
// as 2^(10 - s) + code exactly (the field lands in the mantissa at unit
// weight), so one AND-OR and one subtraction give the code without a shift;
// the scale fields of two sub-blocks are widened as one fp16 pair.  Stores
// are plain shared-memory stores the compiler may schedule (the proxy fence
// after them orders them for the tensor cores).
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

// Q6_K: sub-blocks 2 hf, 2 hf + 1 of chunk cc, weight d * (s - 128) * (q - 32)
// with the scale byte s stored + 128 and the 6-bit code q = low nibble + 16 *
// high pair.  rd / rs / rl / rh: this row's d, scale record, the stage's
// 64-byte unit of the low-nibble record and the high-pair record.
__device__ __forceinline__ void dq_q6k(uint32_t rd, uint32_t rs, uint32_t rl, uint32_t rh, int cc, int hf,
                                       uint4* dst) {
    const __half2 d2 = u2h(g_lds16(rd) * 0x00010001u);
    const int s0 = q16_slot(4 * cc + 2 * hf);   // the two sub-blocks' scale slots s0, s0 + 1
    const uint32_t x = __byte_perm(g_lds32(rs + 4 * (s0 >> 2)), 0u, (s0 & 2) ? 0x4342u : 0x4140u);
    // (1024 + s) - (1024 + 128): the scales minus 128, exact
    const __half2 ap = __hmul2(d2, __hsub2(u2h(x | 0x64006400u), u2h(0x64806480u)));
    const __half2 k1056 = u2h(0x64206420u);   // 1024 + 32
#pragma unroll
    for (int ii = 0; ii < 2; ++ii) {
        const int i = 2 * hf + ii;
        const __half2 a2 = ii ? __high2half2(ap) : __low2half2(ap);
        const uint2 lw = g_lds64(rl + 4 * (4 * i + 2 * (cc & 1)));
        const uint32_t hw = g_lds32(rh + 4 * (4 * i + cc));
        uint32_t o[8];
#pragma unroll
        for (int m = 0; m < 8; ++m) {
            const uint32_t nib = ((m < 4 ? lw.x : lw.y) >> (4 * (m & 3))) & 0x000F000Fu;
            const uint32_t hi2 = (hw >> (2 * m)) & 0x00030003u;
            o[m] = h2u(__hmul2(a2, __hsub2(u2h(nib | (hi2 << 4) | 0x64006400u), k1056)));
        }
        st_row(dst + (2 * i) * kMT, o[0], o[1], o[2], o[3]);
        st_row(dst + (2 * i + 1) * kMT, o[4], o[5], o[6], o[7]);
    }
}

// BF16: the 64-byte record of one 32-weight block (pair p in word 4 (p % 4) +
// p / 4) at rb, converted to fp16 (exact for 2^-14 <= |w| < 65520, to the
// nearest fp16 subnormal below); true if a weight is beyond the fp16 range
__device__ __forceinline__ bool dq_bf16(uint32_t rb, int hf, uint4* dst) {
    uint32_t wd[16];
#pragma unroll
    for (int v = 0; v < 4; ++v) {
        const uint4 q = g_lds128(rb + 16 * v);
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
        st_row(dst + (4 * hf + q) * kMT, o[0], o[1], o[2], o[3]);
    }
    return over;
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
            // columns per stage: a superblock; 128 with a Q8_0 or Q6_K tensor, 64 with a BF16 one
            const bool has32 = f0 == kBF16 || f1 == kBF16;
            const int ks = has32 ? 64 : (f0 == kQ80 || f1 == kQ80 || f0 == kQ6K || f1 == kQ6K) ? 128 : 256;
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
                    const int64_t k0 = (int64_t)st * ks;
                    const int64_t blk = block_len(fz) == 32 ? k0 / 32 : k0 / 256;
                    // Q6_K low nibbles: unit (k0 % 256) / 128 of the record
                    const int64_t uo = (fz == kQ6K && pl == 2) ? ((k0 & 255) >> 7) * (kRowTile * 64) : 0;
                    g_bulk(pk0 + ps * kGPkBytes + doff, src0 + blk * sstep + uo, bytes, pkf + 8 * ps, pol);
                }
            }
            if (bad) { if (lane == 0) fail(); break; }
        }
        // the stages still in flight land before the CTA exits
        for (int q = max(0, pq - kGPk); q < pq; ++q) (void)mbar_wait(pkf + 8 * (q % kGPk), (q / kGPk) & 1);
    } else if (warp == kWarpB) {
        // ---- activations: the chunk's rows of the unit's tile, one bulk copy
        // (its eight 8-column pieces are contiguous in the tile-ordered copy)
        // into the operand slot; the MMA reads rows N .. Npad - 1 of a piece
        // from the next piece or past the copied run: they only reach
        // accumulator columns the epilogue never reads
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
                // the chunk's eight pieces are one contiguous run of 8 N x 16
                // bytes; the MMA's B descriptor steps N x 16 bytes per piece
                if (lane == 0) {
                    g_arrive_tx(opf + 8 * s, (uint32_t)(U.N * 128));
                    asm volatile("cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];"
                                 ::"r"(ring + s * kGSlotBytes + kBOfs), "l"(src + perm_piece(U.r0, K, U.N, c * 8, 0)),
                                   "r"((uint32_t)(U.N * 128)), "r"(opf + 8 * s) : "memory");
                }
                __syncwarp();
            }
            if (bad) { if (lane == 0) fail(); break; }
            __syncwarp();
            if (lane == 0) mbar_arrive(ue + 8 * us);
        }
    } else if (warp == kWarpM) {
        // ---- MMA issue.  The A descriptors of the slots are built once, B's
        // per unit: B holds the chunk's eight pieces of N rows x 16 bytes one
        // after the other (leading byte offset N x 16).  A 16-column step of K
        // moves A by 2 * kMT * 16 bytes and B by 2 * N * 16 bytes, i.e. the
        // descriptors' start-address field (bytes / 16) by 256 and 2 N.
        uint64_t dA[kGOpsMax][2], dB[kGOpsMax];
#pragma unroll
        for (int sl2 = 0; sl2 < kGOpsMax; ++sl2) {
            const uint32_t sbase = ring + sl2 * kGSlotBytes;
            dA[sl2][0] = sdesc(sbase, kMT * 16, 128);
            dA[sl2][1] = sdesc(sbase + kABytes, kMT * 16, 128);
        }
        int mq = 0, last = -1;
        for (int ui = 0;; ++ui) {
            const int us = ui & 1;
            if (!mbar_wait(uf + 8 * us, (ui >> 1) & 1)) { if (lane == 0) fail(); break; }
            const GUnit U = s_unit[us];
            if (U.u < 0) break;
#pragma unroll
            for (int sl2 = 0; sl2 < kGOpsMax; ++sl2)
                dB[sl2] = sdesc(ring + sl2 * kGSlotBytes + kBOfs, (uint32_t)U.N * 16u, 128);
            const uint32_t bstep = 2u * (uint32_t)U.N;
            bool bad = false;
            for (int c = 0; c < nC; ++c, ++mq) {
                const int s = mq % kGOps;
                if (!mbar_wait(opf + 8 * s, (mq / kGOps) & 1)) { bad = true; break; }
                if (lane == 0) {
                    // (the workers fenced their operand stores; the activations came by bulk copy)
                    asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
                    const uint32_t idesc = idesc_f16(kMT, U.Npad);
                    uint64_t a0 = dA[0][0], a1 = dA[0][1], b0 = dB[0];
#pragma unroll
                    for (int q = 1; q < kGOpsMax; ++q)
                        if (s == q) { a0 = dA[q][0]; a1 = dA[q][1]; b0 = dB[q]; }
#pragma unroll
                    for (int kk = 0; kk < kKC / 16; ++kk) {
                        const uint32_t acc = (c > 0 || kk > 0) ? 1u : 0u;
                        mma_f16(tbase, a0 + 256u * kk, b0 + bstep * kk, idesc, acc);
                        if (!kDown) mma_f16(tbase + kGNT, a1 + 256u * kk, b0 + bstep * kk, idesc, acc);
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
        const int z = kDown ? 0 : (warp >> 3);
        const int gsel = kDown ? (warp >> 3) : 0;
        const int tl = warp & 3, hf = (warp >> 2) & 1;
        const int rr = 32 * tl + lane;
        uint4* const sv4 = reinterpret_cast<uint4*>(smem);
        bool w_over = false;        // a BF16 weight of this thread's rows beyond the fp16 range
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
            // one chunk: c its index in the unit, cc its 64-column quarter of the
            // superblock, lb its first Q8_0 / BF16 block in the stage
            // (kKq: a unit of K-quant tensors only, whose stages are whole superblocks)
            auto chunk = [&](auto kKq, int c, int cc, int lb, uint32_t so) -> bool {
                const int g = gbase + c, s = g % kGOps;
                if (g >= kGOps && !mbar_wait(ope + 8 * s, ((g - kGOps) / kGOps) & 1)) return false;
                if (failed()) return false;
                uint4* const dst = sv4 + (s * kGSlotBytes + z * kABytes) / 16 + rr;
                if (fz == kQ2K) {
                    dq_q2k(B, cc, hf, dst);
                } else if (fz == kQ3K) {
                    dq_q3k(B, cc, hf, dst);
                } else if (decltype(kKq)::value || fz == kQ4K) {
                    dq_q4k(B, cc, hf, dst);
                } else if (fz == kQ80) {   // block lb + hf of the stage
                    const uint32_t cp = rec[1] + so + (lb + hf) * (32 * 32);
                    const uint4 w0 = g_lds128(cp), w1 = g_lds128(cp + 16);
                    const uint32_t w[8] = {w0.x, w0.y, w0.z, w0.w, w1.x, w1.y, w1.z, w1.w};
                    dq_q80(w, g_lds16(rec[0] + so + (lb + hf) * (32 * 2)), hf, dst);
                } else if (fz == kQ6K) {
                    dq_q6k(rec[0] + so, rec[1] + so, rec[2] + so, rec[3] + so, cc, hf, dst);
                } else {   // BF16: block lb + hf of the stage
                    w_over |= dq_bf16(rec[0] + so + (lb + hf) * (32 * 64), hf, dst);
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
                if (fz == kQ2K || fz == kQ3K || fz == kQ4K) {   // (the others read their fields per chunk)
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
                        if (!chunk(std::true_type{}, c, cl, 0, so)) { bad = true; break; }
                    }
                } else {
                    // 128 or 64 columns (a Q8_0, Q6_K or BF16 tensor in the unit)
                    for (int cl = 0; cl < cps; ++cl) {
                        const int c = cps * st + cl;
                        if (c >= nC) break;
                        if (kDown && (c & 1) != gsel) continue;
                        if (!chunk(std::false_type{}, c, c & 3, 2 * cl, so)) { bad = true; break; }
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
        if (w_over) atomicOr(A.err, kErrWeightRange);
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
    cudaFuncSetAttribute(gemm_ws_kernel<false>, cudaFuncAttributeMaxDynamicSharedMemorySize, g_smem(false));
    cudaFuncSetAttribute(gemm_ws_kernel<true>, cudaFuncAttributeMaxDynamicSharedMemorySize, g_smem(true));
}

}  // namespace

cudaError_t launch_prefill(const Dims& d, const ExpertTab& tab, const Work& w, float* out, cudaStream_t s) {
    if (d.T == 0) return cudaSuccess;
    const int g_psms = device_setup(kSetupPrefill, prefill_setup);
    if (g_psms <= 0) return cudaErrorInvalidDevice;
    PrefillArgs A;
    A.d = d;
    A.offsets = w.offsets; A.perm = w.perm; A.active = w.active; A.wts = w.wts;
    A.x16 = w.x16; A.xe = w.xe; A.h16 = w.h16; A.pdn = w.pdn; A.err = w.err;
    A.next = w.counters;
    A.xp = reinterpret_cast<uint8_t*>(w.pdn);   // dead until the down GEMM writes its partial rows
    prof_begin("xperm", s);
    cudaError_t err = launch_pdl(xperm_kernel, dim3(4 * g_psms), dim3(kXpWarps * 32), 0, s,
                                 static_cast<const __half*>(w.x16), static_cast<const int32_t*>(w.offsets),
                                 static_cast<const int32_t*>(w.perm), static_cast<const int32_t*>(w.active), d, A.xp);
    prof_end(s);
    if (err != cudaSuccess) return err;
    prof_begin("gateup_tc", s);
    err = launch_pdl(gemm_ws_kernel<false>, dim3(g_psms), dim3(g_threads(false)), g_smem(false), s, tab, A);
    prof_end(s);
    if (err != cudaSuccess) return err;
    prof_begin("down_tc", s);
    err = launch_pdl(gemm_ws_kernel<true>, dim3(g_psms), dim3(g_threads(true)), g_smem(true), s, tab, A);
    prof_end(s);
    if (err != cudaSuccess) return err;
    return launch_combine(d, w.pdn, out, s);
}

}  // namespace mq
