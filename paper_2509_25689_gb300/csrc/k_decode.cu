// Expert FFN kernel for decode-sized batches (arXiv 2509.25689 Fig. 1: a
// shared expert plus router-weighted routed SwiGLU experts; each expert
// tensor stored in its own k-quant style block format, Sec. 3.3).
//
// Dequant-fused GEMV on the legacy tensor-core path (mma.sync m16n8k16,
// fp16 x fp16 -> fp32):
//   A (16 rows x 16 k) = weight codes read straight from the packed words:
//     one AND per code pair leaves the code in the mantissa of an fp16
//     subnormal (value code * 2^(s-24), s a positional power of two that the
//     activation carries inverted);
//   B (16 k x 8 cols) = the prepared activation (mq_actprep.cuh), column n
//     carrying sub-block n of an 8-sub-block group and zero elsewhere, fixed
//     per lane so nothing is masked in the loop;
//   D (16 rows x 8 cols) = per-(row, sub-block) partial dot products, so the
//     sub-block scales and mins are applied once per tile in fp32.
// One persistent kernel runs the whole expert FFN of a call.  Work is cut
// into items claimed from one per-call counter in this order: the shared
// expert's gate/up items (they need no routing result and start while the
// routing kernel runs), the routed experts' gate/up items, the shared
// expert's down items, the routed experts' down items.  A gate/up item is 32
// rows x all superblocks of gate and of up, a down item two 32-row blocks x
// all superblocks, of one expert x up to 4 tokens.  The SwiGLU output h of an
// expert slot is published per 32-row block (the item's finisher writes it,
// fences, and increments the slot's counter); a down item's producer streams
// its weights at once and copies h only when the slot's counter says every
// block is in, so down items of the first experts overlap the last gate/up
// items and no CTA idles at a kernel boundary.  Every gate/up item is claimed
// before any down item, so each awaited block is held by a CTA that finishes
// it without waiting on anything.
// The packed layout keeps any superblock range of a 32-row tile contiguous in
// every plane, so a dedicated producer warp streams each item through a
// shared-memory ring with 1D bulk (TMA) copies that complete on mbarriers; the
// consumer warps (all 32 rows x every kCols-th superblock of a stage each,
// the columns rotated from stage to stage) run the tensor-core math.  At the
// end of an item the CTA reduces its warps' sums in a fixed order (SwiGLU and
// the prepared h for gate/up, one partial output row block per assignment
// for down), so results are deterministic.  Every wait (mbarriers, the h
// counters) is bounded (about 1 s) and reports to an error word.
#include <cuda_fp16.h>

#include "mq_actprep.cuh"
#include "mq_internal.h"

namespace mq {
namespace {

constexpr unsigned kFull = 0xffffffffu;

__device__ __forceinline__ void mma16816(float (&d)[4], uint32_t a0, uint32_t a1, uint32_t a2, uint32_t a3,
                                         uint32_t b0, uint32_t b1) {
    asm("mma.sync.aligned.m16n8k16.row.col.f32.f16.f16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, {%0,%1,%2,%3};"
        : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
        : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1));
}

// bf16 x bf16 -> fp32 (the BF16 weight tiles)
__device__ __forceinline__ void mma16816_bf16(float (&d)[4], uint32_t a0, uint32_t a1, uint32_t a2, uint32_t a3,
                                              uint32_t b0, uint32_t b1) {
    asm("mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, {%0,%1,%2,%3};"
        : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
        : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1));
}

__device__ __forceinline__ float h2f(uint32_t bits16) { return __half2float(__ushort_as_half((unsigned short)bits16)); }

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
// Bounded wait: gives up after `limit_ns` (1 s unless a test shortened it),
// records `code` in the error word.
__device__ __forceinline__ bool mbar_wait(uint32_t bar, uint32_t parity, uint32_t* err, uint32_t code,
                                          uint64_t limit_ns) {
    if (mbar_try(bar, parity)) return true;
    const uint64_t t0 = global_ns();
    for (;;) {
        if (mbar_try(bar, parity)) return true;
        if (global_ns() - t0 > limit_ns) { atomicOr(err, code); return false; }
    }
}
__device__ __forceinline__ void bulk_copy(uint32_t dst, const void* src, uint32_t bytes, uint32_t bar) {
    asm volatile("cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];"
                 ::"r"(dst), "l"(src), "r"(bytes), "r"(bar) : "memory");
}
__device__ __forceinline__ uint64_t evict_first_policy() {
    uint64_t p;
    asm volatile("createpolicy.fractional.L2::evict_first.b64 %0, 1.0;" : "=l"(p));
    return p;
}
__device__ __forceinline__ void bulk_copy_hint(uint32_t dst, const void* src, uint32_t bytes, uint32_t bar, uint64_t pol) {
    asm volatile("cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes.L2::cache_hint [%0], [%1], %2, [%3], %4;"
                 ::"r"(dst), "l"(src), "r"(bytes), "r"(bar), "l"(pol) : "memory");
}
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

#ifndef MQ_DECODE_CONSUMERS
#define MQ_DECODE_CONSUMERS 8
#endif
#ifndef MQ_DECODE_SLOTS
#define MQ_DECODE_SLOTS 4
#endif
constexpr int kConsumers = MQ_DECODE_CONSUMERS;     // consumer warps
constexpr int kNT = kConsumers >= 16 ? 1 : 2;       // 16-row MMA tiles per warp (of the stage's two)
constexpr int kCols = kConsumers * kNT / 2;         // superblock columns the warps are spread over
constexpr int kThreads = (kConsumers + 1) * 32;     // + one producer warp
constexpr int kProducerWarp = kConsumers;
// Ring of kNST slots (one-token kernel 4 x 48 KB: Q3_K down stages are
// 37 KB, Q2_K gate/up stages of 14 superblocks 47 KB, Q8_0 stages of 5
// superblocks 44 KB; several-token kernel 4 x 46 KB, which leaves room for
// its second item-end reduction buffer)
constexpr int kNST = MQ_DECODE_SLOTS;
__host__ __device__ constexpr int ring_bytes(int mt) { return mt == 1 ? 192 * 1024 : 184 * 1024; }
__host__ __device__ constexpr int slot_bytes(int mt) { return ring_bytes(mt) / kNST; }
constexpr int kStageSb = 16;                        // superblocks per stage (Q8_0: 8), fewer if over budget
constexpr int kMaxCachedAssign = 1024;              // routed assignments cached in smem
#ifndef MQ_SPLIT_SHARED
#define MQ_SPLIT_SHARED 1
#endif
#ifndef MQ_PREROUTE_DEPTH
#define MQ_PREROUTE_DEPTH 3
#endif
constexpr int kPreRouteDepth = MQ_PREROUTE_DEPTH;   // stages in flight before the routing result is in
static_assert(kPreRouteDepth >= 1 && kPreRouteDepth <= kNST, "pre-routing depth");
constexpr uint32_t kErrFull = 1u, kErrEmpty = 2u, kErrReady = 32u;
// named barrier 1: the consumer warps only
__device__ __forceinline__ void consumer_sync() { asm volatile("bar.sync 1, %0;" ::"n"(kConsumers * 32) : "memory"); }
__device__ __forceinline__ uint32_t ld_acquire(const uint32_t* p) {
    uint32_t v;
    asm volatile("ld.acquire.gpu.global.u32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
    return v;
}
__device__ __forceinline__ void red_release_add(uint32_t* p, uint32_t v) {
    asm volatile("red.release.gpu.global.add.u32 [%0], %1;" ::"l"(p), "r"(v) : "memory");
}
__device__ __forceinline__ uint32_t atom_acq_rel_add(uint32_t* p, uint32_t v) {
    uint32_t old;
    asm volatile("atom.acq_rel.gpu.global.add.u32 %0, [%1], %2;" : "=r"(old) : "l"(p), "r"(v) : "memory");
    return old;
}

// stage header written by the producer (one per ring slot); the stage's
// byte layout is geo[down][fmt - 1][ntok - 1]
struct __align__(16) Hdr {
    int32_t item, j, nst, s0;
    int32_t ks, fmt, tensor, ntok;   // tensor: 0 gate, 1 up, 2 down rows rb, 3 down rows rb + 1
    int32_t rb, e, shared, slot;
    int32_t asg[kDecodeTok];
    int32_t kb, half, pad0, pad1;      // first superblock of the item's K range; K half (-1: whole K)
};

// token pieces in a stage: the family fragments and the per-superblock
// statistics, each for the stage's ks superblocks
struct TokLay { int x, s, stride; };
// (BF16: the bf16 hi and lo operands of the token instead)
__host__ __device__ __forceinline__ TokLay tok_lay(int fmt, int ks) {
    TokLay t;
    int at = 0;
    t.x = at; at += ks * 512;
    t.s = at; at += ks * (fmt == kBF16 ? 512 : kStatFloats * 4);
    t.stride = (at + 127) & ~127;
    return t;
}

__host__ __device__ __forceinline__ int weight_stage_bytes(int fmt, int ks) {
    const PlaneBytes pb = plane_bytes(fmt);
    const int nblk = block_len(fmt) == 32 ? 8 * ks : ks;
    int at = 0;
    for (int p = 0; p < pb.n; ++p) at += (32 * nblk * pb.b[p] + 127) & ~127;
    return at;
}
// superblocks per stage for a format and token count (fits a ring slot)
__host__ __device__ __forceinline__ int stage_sb(int fmt, int ntok, int stage_bytes) {
    int ks = fmt == kQ80 ? kStageSb / 2 : fmt == kBF16 ? 2 : kStageSb;
    while (ks > 1 && weight_stage_bytes(fmt, ks) + ntok * tok_lay(fmt, ks).stride > stage_bytes) --ks;
    return ks;
}

// per-CTA cache of the routing result: slot -> expert, first entry, tokens,
// and the items before each slot (gate/up and down)
struct SlotCache {
    int32_t e[kMaxExperts + 1], first[kMaxExperts + 1], ntot[kMaxExperts + 1];
    int32_t pre_gu[kMaxExperts + 2], pre_dn[kMaxExperts + 2];
    // the slot's tensors and formats (gate, up, down), copied from the expert
    // table once: a kernel-parameter lookup with a run-time index goes
    // through the constant cache, which the kernel's instructions share
    const uint8_t* p[kMaxExperts + 1][3];
    uint8_t fmt[kMaxExperts + 1][3];
};

// Stage geometry of one (kind, format, tokens per item), computed once per
// launch on the host so the producer does no layout arithmetic per stage.
struct Geo {
    int32_t pl[4];       // plane starts in the tensor
    int32_t rbstr[4];    // bytes per 32-row block in each plane
    int32_t woff[4], cstr[4];  // plane regions in the stage, bytes per superblock
    int32_t tok0, tstride, tx, ts;   // token pieces: first byte, bytes per token, fragments, statistics
    int16_t per, nst, npl, pad;      // superblocks per stage, stages per tensor, planes
};
static_assert(sizeof(Geo) == 88, "geometry record");

__host__ __device__ inline void make_geo(Geo& G, const Dims& d, bool down, int fmt, int ntok, int slot_b) {
    const int nsb = down ? (d.I + 255) / 256 : (d.H + 255) / 256;
    const TensorLayout L = tensor_layout(fmt, down ? d.H : d.I, down ? d.I : d.H);
    const PlaneBytes pb = plane_bytes(fmt);
    const int bmul = block_len(fmt) == 32 ? 8 : 1;   // Q8_0 / BF16: 8 blocks of 32 per superblock
    G.per = (int16_t)stage_sb(fmt, ntok, slot_b);
    G.nst = (int16_t)((nsb + G.per - 1) / G.per);
    G.npl = (int16_t)pb.n;
    int at = 0;
    for (int pl = 0; pl < 4; ++pl) {
        G.woff[pl] = at;
        G.cstr[pl] = pl < pb.n ? 32 * bmul * pb.b[pl] : 0;
        G.pl[pl] = (int32_t)L.plane[pl];
        G.rbstr[pl] = pl < pb.n ? (int32_t)(L.blocks_per_row * 32 * pb.b[pl]) : 0;
        if (pl < pb.n) at += (32 * bmul * G.per * pb.b[pl] + 127) & ~127;
    }
    const TokLay tl = tok_lay(fmt, G.per);
    G.tok0 = at; G.tstride = tl.stride; G.tx = tl.x; G.ts = tl.s;
    G.pad = 0;
}

struct DecodeArgs {
    Dims d;
    int nsbx, nsbi;          // superblocks along hidden / inter
    const __half* xq; const float* xs;   // prepared tokens
    __half* hq; float* hs;               // prepared SwiGLU outputs (per assignment)
    const int32_t* perm; const float* wts;
    const Plan* plan;
    float* pdn;              // [A][H]
    uint32_t* next;          // item counter
    uint32_t* hready;        // [kMaxExperts + 1] per slot: published h blocks (tokens x 32-row blocks)
    uint32_t* scount;        // [T][I / 32] halves of a shared gate/up block finished (K split)
    float* spart;            // [T][2 halves][2 (gate, up)][I] the halves' sums
    const uint32_t* logits_done;   // logits CTAs done (their prepared tokens are written)
    const uint32_t* route_ready;   // non-zero once the routing result is written
    uint32_t n_logit_ctas;
    uint32_t* err;
    uint64_t wait_ns;        // limit of every bounded wait
    int fail_first_stage;    // test hook: the producer posts nothing for its first stage
    int split_shared;        // the shared expert's gate/up blocks are split in two K halves
    Geo geo[2][kNumFormats][kDecodeTok];   // [down][format][tokens], computed on the host
};

struct ItemDesc {            // decoded item (producer side)
    int e, rb, tg, ntok, shared, nst0, nst, down, slot;
    int kb, ke, half;        // superblock range [kb, ke) of K; half of a split item (-1: whole K)
    int vec[kDecodeTok], asg[kDecodeTok];
};

// Item id -> slot, rows, tokens.  Ids [0, n_gu) are gate/up items, [n_gu,
// n_gu + n_dn) down items; both in slot order (the shared expert first).
__device__ __forceinline__ void decode_item(const DecodeArgs& A, const SlotCache& sc, const int32_t* s_perm,
                                            int n_slots, int n_gu, int id, int& cur_gu, int& cur_dn,
                                            ItemDesc& it) {
    const bool down = id >= n_gu;
    const int32_t* pre = down ? sc.pre_dn : sc.pre_gu;
    const int lid = down ? id - n_gu : id;
    int& cursor = down ? cur_dn : cur_gu;   // ids grow, so each walk only moves forward
    while (cursor + 1 < n_slots && pre[cursor + 1] <= lid) ++cursor;
    const int p = cursor;
    it.slot = p;
    it.down = down ? 1 : 0;
    int local = lid - pre[p];
    const Dims& d = A.d;
    // gate/up items: one 32-row block of gate and up; down items: two 32-row blocks.
    // The shared expert's gate/up blocks are split in two K halves (two items,
    // the halves of a block claimed one after the other), so that every CTA has
    // shared-expert work while the routing result is computed.
    const int nrb = down ? d.H / 64 : d.I / 32;
    const int nsb = down ? A.nsbi : A.nsbx;
    it.half = -1; it.kb = 0; it.ke = nsb;
    if (!down && p < d.has_shared && A.split_shared) {
        it.half = local & 1;
        local >>= 1;
        const int mid = nsb / 2;
        it.kb = it.half ? mid : 0;
        it.ke = it.half ? nsb : mid;
    }
    it.tg = local / nrb;
    it.rb = (local - it.tg * nrb) * (down ? 2 : 1);
    it.e = sc.e[p];
    it.shared = p < d.has_shared;
    it.ntok = min(kDecodeTok, sc.ntot[p] - it.tg * kDecodeTok);
#pragma unroll
    for (int j = 0; j < kDecodeTok; ++j) {
        int t = 0, a = 0;
        if (j < it.ntok) {
            const int q = it.tg * kDecodeTok + j;
            if (it.shared) { t = q; a = d.T * d.K + q; }
            else {
                const int idx = sc.first[p] + q;
                a = idx < kMaxCachedAssign ? s_perm[idx] : __ldcg(A.perm + idx);
                t = a / d.K;
            }
        }
        it.asg[j] = a;
        it.vec[j] = down ? a : t;
    }
    it.nst0 = 0;
    it.nst = 0;
}

// ---- consumer math: one warp = the 32 rows of the stage (two 16-row MMA
// tiles) x one superblock (Q8_0: half of its code pairs) x one token.
//
// MMA m16n8k16, rows g / g+8 of a tile for lane (g, t).  One MMA covers pair
// m of eight sub-blocks: lane t feeds sub-block t of the group through a0/a1
// and sub-block t+4 through a2/a3, so column n of B (and D) is sub-block n
// of the group.  Operand B is static per lane: lane (g, t) supplies
// activations only where g == t (b0) or g == t + 4 (b1) and zeros otherwise,
// so no masking happens in the loop; the zero lanes read a zero block of
// shared memory.  Both row tiles share the B registers.  D lane (g, t) then
// holds sub-blocks 2t, 2t+1 of the group, whose scale fields are one word of
// the slot-ordered record.  acc[2 * tile + h] accumulates row 16 tile + g + 8 h.
__device__ __forceinline__ uint32_t sub4(uint4 v, int i) { return i == 0 ? v.x : i == 1 ? v.y : i == 2 ? v.z : v.w; }
__device__ __forceinline__ float u8f(uint32_t w, int b) { return (float)((w >> (8 * b)) & 0xffu); }
__device__ __forceinline__ void ld_frag8(uint32_t a, uint32_t (&X)[8]) {
    const uint4 u = lds128(a), v = lds128(a + 16);
    X[0] = u.x; X[1] = u.y; X[2] = u.z; X[3] = u.w; X[4] = v.x; X[5] = v.y; X[6] = v.z; X[7] = v.w;
}

// A tile's MMA sums: [tile][sub-block group][pair parity][D fragment]
// (Q2_K / Q3_K: the two sub-block groups; Q4_K / Q8_0: four accumulators
// of the same sums, added in the epilogue).
template <int NT> struct TileAcc { float DD[NT][2][2][4]; };

// Loads one (superblock, token) tile of the warp's rows and issues its MMAs
// into T; tile_epi applies the scales once the sums are in.
template <int FMT, int NT>
__device__ __forceinline__ void tile_mma(const Geo& h, uint32_t st, int jj, int half, int rt0, int tk,
                                         uint32_t zaddr, TileAcc<NT>& T) {
    // rows of this warp: i = 0 .. 2 NT - 1 -> row 16 (rt0 + i / 2) + 8 (i % 2) + g
    constexpr int NR = 2 * NT;
    const int lane = threadIdx.x & 31, g = lane >> 2, t = lane & 3;
    const bool own0 = g == t, own1 = g == t + 4;
    const int w1 = h.woff[1], w2 = h.woff[2], w3 = h.woff[3];
    const uint32_t tb = st + h.tok0 + tk * h.tstride;
    const uint32_t xb = tb + h.tx + jj * 512;
    const int rbase = jj * 32 + 16 * rt0 + g;   // record index of this lane's first row
    auto rec_of = [&](int i) { return rbase + 16 * (i >> 1) + 8 * (i & 1); };
#pragma unroll
    for (int i = 0; i < NT * 16; ++i) (&T.DD[0][0][0][0])[i] = 0.0f;

    // Issue order: every MMA of a step goes to a different accumulator and an
    // accumulator is reused only 8 MMAs later, so the in-order warp does not
    // stall on the MMA latency inside a tile (all B fragments are loaded first).
    if (FMT == kQ2K || FMT == kQ3K) {
        const uint32_t cp = FMT == kQ2K ? w3 : w2;   // 2-bit code plane
        uint4 c[NR];
        uint2 hv[NR];
#pragma unroll
        for (int i = 0; i < NR; ++i) {
            c[i] = lds128(st + cp + rec_of(i) * 64 + 16 * t);
            if (FMT == kQ3K) hv[i] = lds64(st + w3 + rec_of(i) * 32 + 8 * t);
        }
        uint32_t XA[2][8], XB[2][8];
#pragma unroll
        for (int gm = 0; gm < 2; ++gm) {
            ld_frag8(own0 ? xb + 32 * (8 * gm + t) : zaddr, XA[gm]);
            ld_frag8(own1 ? xb + 32 * (8 * gm + 4 + t) : zaddr, XB[gm]);
        }
        uint32_t qa[2][NR], qb[2][NR], sa[2][NR], sbb[2][NR];   // per row: sub-blocks t (a0/a1) and t+4 (a2/a3)
#pragma unroll
        for (int gm = 0; gm < 2; ++gm)
#pragma unroll
            for (int i = 0; i < NR; ++i) {
                qa[gm][i] = sub4(c[i], 2 * gm); qb[gm][i] = sub4(c[i], 2 * gm + 1);
                sa[gm][i] = qa[gm][i] >> 10; sbb[gm][i] = qb[gm][i] >> 10;
            }
        if (FMT == kQ2K) {
#pragma unroll
            for (int m = 0; m < 8; ++m) {
                const uint32_t mk = 0x00030003u << (m <= 4 ? 2 * m : 2 * (m - 5));
                const bool sh = m > 4;
#pragma unroll
                for (int gm = 0; gm < 2; ++gm)
#pragma unroll
                    for (int tl = 0; tl < NT; ++tl)
                        mma16816(T.DD[tl][gm][m & 1], (sh ? sa[gm][2 * tl] : qa[gm][2 * tl]) & mk,
                                 (sh ? sa[gm][2 * tl + 1] : qa[gm][2 * tl + 1]) & mk,
                                 (sh ? sbb[gm][2 * tl] : qb[gm][2 * tl]) & mk,
                                 (sh ? sbb[gm][2 * tl + 1] : qb[gm][2 * tl + 1]) & mk, XA[gm][m], XB[gm][m]);
            }
        } else {
            // Q3_K: code = low2 + 4 hbit.  The low two bits go through the same
            // MMAs as Q2_K; the high bits get MMAs of their own into the same
            // accumulators: the high bit of pair m sits at bit m (and 16 + m)
            // of its half of the hmask word (the second sub-block of a word one
            // byte up, shifted down once), so one AND makes an fp16 pair
            // hbit * 2^(m-24), and the activation operand is scaled by
            // 4 * 2^(pos(m) - m) (exact powers of two) to weigh it 4 x.
            uint32_t ha[2][NR], hb[2][NR];
#pragma unroll
            for (int gm = 0; gm < 2; ++gm)
#pragma unroll
                for (int i = 0; i < NR; ++i) { ha[gm][i] = gm ? hv[i].y : hv[i].x; hb[gm][i] = ha[gm][i] >> 8; }
#pragma unroll
            for (int m = 0; m < 8; ++m) {
                const uint32_t mk = 0x00030003u << (m <= 4 ? 2 * m : 2 * (m - 5));
                const bool sh = m > 4;
#pragma unroll
                for (int gm = 0; gm < 2; ++gm)
#pragma unroll
                    for (int tl = 0; tl < NT; ++tl)
                        mma16816(T.DD[tl][gm][m & 1], (sh ? sa[gm][2 * tl] : qa[gm][2 * tl]) & mk,
                                 (sh ? sa[gm][2 * tl + 1] : qa[gm][2 * tl + 1]) & mk,
                                 (sh ? sbb[gm][2 * tl] : qb[gm][2 * tl]) & mk,
                                 (sh ? sbb[gm][2 * tl + 1] : qb[gm][2 * tl + 1]) & mk, XA[gm][m], XB[gm][m]);
            }
#pragma unroll
            for (int m = 0; m < 8; ++m) {
                const uint32_t mh = 0x00010001u << m;
                // 4 * 2^(pos(m) - m): 2^(m+2) for m <= 4, 2^(m-8) above (fp16 bits)
                const int e = m <= 4 ? m + 2 : m - 8;
                const uint32_t sc16 = (uint32_t)(15 + e) << 10;
                const __half2 scl = __halves2half2(__ushort_as_half((unsigned short)sc16), __ushort_as_half((unsigned short)sc16));
#pragma unroll
                for (int gm = 0; gm < 2; ++gm) {
                    const __half2 xa = __hmul2(*reinterpret_cast<const __half2*>(&XA[gm][m]), scl);
                    const __half2 xb2 = __hmul2(*reinterpret_cast<const __half2*>(&XB[gm][m]), scl);
                    const uint32_t ua = *reinterpret_cast<const uint32_t*>(&xa), ub = *reinterpret_cast<const uint32_t*>(&xb2);
#pragma unroll
                    for (int tl = 0; tl < NT; ++tl)
                        mma16816(T.DD[tl][gm][(m + 1) & 1], ha[gm][2 * tl] & mh, ha[gm][2 * tl + 1] & mh,
                                 hb[gm][2 * tl] & mh, hb[gm][2 * tl + 1] & mh, ua, ub);
                }
            }
        }
    } else if (FMT == kQ4K) {
        // pairs 8 hm + mm accumulate into group slot hm (the epilogue adds both)
        uint4 cA[NR], cB[NR];   // rows: sub-blocks t (unit 0) and t+4 (unit 1)
#pragma unroll
        for (int i = 0; i < NR; ++i) {
            const int r = rec_of(i) - jj * 32;
            cA[i] = lds128(st + w3 + ((jj * 2 + 0) * 32 + r) * 64 + 16 * t);
            cB[i] = lds128(st + w3 + ((jj * 2 + 1) * 32 + r) * 64 + 16 * t);
        }
        uint32_t XA[2][8], XB[2][8];
#pragma unroll
        for (int hm = 0; hm < 2; ++hm) {
            ld_frag8(own0 ? xb + 64 * t + 32 * hm : zaddr, XA[hm]);
            ld_frag8(own1 ? xb + 64 * (t + 4) + 32 * hm : zaddr, XB[hm]);
        }
#pragma unroll
        for (int mm = 0; mm < 8; ++mm) {
#pragma unroll
            for (int hm = 0; hm < 2; ++hm) {
                const int m = 8 * hm + mm, wi = m >> 2, j = m & 3;
                const uint32_t mk = (j & 1) ? 0x00F000F0u : 0x000F000Fu;
                const int sh = j < 2 ? 0 : 8;
#pragma unroll
                for (int tl = 0; tl < NT; ++tl)
                    mma16816(T.DD[tl][hm][mm & 1], (sub4(cA[2 * tl], wi) >> sh) & mk,
                             (sub4(cA[2 * tl + 1], wi) >> sh) & mk, (sub4(cB[2 * tl], wi) >> sh) & mk,
                             (sub4(cB[2 * tl + 1], wi) >> sh) & mk, XA[hm][mm], XB[hm][mm]);
            }
        }
    } else if (FMT == kQ6K) {
        // q = low nibble + 16 * high two bits.  Nibble MMAs as Q4_K's (operand
        // family F4: pair m carries 2^(4 (m & 1))) on 16-wide sub-blocks; the
        // high two bits sit in the Q2_K code order and go into the same
        // accumulators weighed by 16: each pair's field is moved by one of
        // three shifts of its word (<< 4, none, >> 6) to a bit position p
        // <= 8 of its fp16 half, and the F4 operand is scaled by the exact
        // power of two 2^(4 + 4 (m & 1) - p) (at most 2^2 / 2^6 for even / odd
        // m, which the F4 range leaves room for).
        uint4 n0[NR], n1[NR], c[NR];   // nibbles: unit 0 (sub-blocks t, t+4), unit 1 (t+8, t+12); high bits
#pragma unroll
        for (int i = 0; i < NR; ++i) {
            const int r = rec_of(i) - jj * 32;
            n0[i] = lds128(st + w2 + ((jj * 2 + 0) * 32 + r) * 64 + 16 * t);
            n1[i] = lds128(st + w2 + ((jj * 2 + 1) * 32 + r) * 64 + 16 * t);
            c[i] = lds128(st + w3 + rec_of(i) * 64 + 16 * t);
        }
        uint32_t XA[2][8], XB[2][8];
#pragma unroll
        for (int gm = 0; gm < 2; ++gm) {
            ld_frag8(own0 ? xb + 32 * (8 * gm + t) : zaddr, XA[gm]);
            ld_frag8(own1 ? xb + 32 * (8 * gm + 4 + t) : zaddr, XB[gm]);
        }
#pragma unroll
        for (int m = 0; m < 8; ++m) {
            const uint32_t mk = (m & 1) ? 0x00F000F0u : 0x000F000Fu;
            const int sh = (m & 2) ? 8 : 0;
            const int wi = m >> 2;   // word of the pair within a sub-block's two
#pragma unroll
            for (int gm = 0; gm < 2; ++gm)
#pragma unroll
                for (int tl = 0; tl < NT; ++tl) {
                    const uint4& ua = gm ? n1[2 * tl] : n0[2 * tl];
                    const uint4& ub = gm ? n1[2 * tl + 1] : n0[2 * tl + 1];
                    mma16816(T.DD[tl][gm][m & 1], (sub4(ua, wi) >> sh) & mk, (sub4(ub, wi) >> sh) & mk,
                             (sub4(ua, 2 + wi) >> sh) & mk, (sub4(ub, 2 + wi) >> sh) & mk, XA[gm][m], XB[gm][m]);
                }
        }
#pragma unroll
        for (int m = 0; m < 8; ++m) {
            // word shift (left 4 / none / right 6), resulting bit position, operand scale 2^e
            const int shl = m <= 1 ? 4 : 0, shr = m >= 5 ? 6 : 0;
            const int pos = 2 * m + shl - shr;
            const int e = 4 + 4 * (m & 1) - pos;
            const uint32_t mk = 0x00030003u << pos;
            const uint32_t sc16 = (uint32_t)(15 + e) << 10;
            const __half2 scl = __halves2half2(__ushort_as_half((unsigned short)sc16), __ushort_as_half((unsigned short)sc16));
#pragma unroll
            for (int gm = 0; gm < 2; ++gm) {
                uint32_t ua = XA[gm][m], ub = XB[gm][m];
                if (e != 0) {
                    const __half2 xa = __hmul2(*reinterpret_cast<const __half2*>(&ua), scl);
                    const __half2 xb2 = __hmul2(*reinterpret_cast<const __half2*>(&ub), scl);
                    ua = *reinterpret_cast<const uint32_t*>(&xa);
                    ub = *reinterpret_cast<const uint32_t*>(&xb2);
                }
#pragma unroll
                for (int tl = 0; tl < NT; ++tl) {
                    const uint32_t qa0 = sub4(c[2 * tl], 2 * gm), qa1 = sub4(c[2 * tl + 1], 2 * gm);
                    const uint32_t qb0 = sub4(c[2 * tl], 2 * gm + 1), qb1 = sub4(c[2 * tl + 1], 2 * gm + 1);
                    mma16816(T.DD[tl][gm][(m + 1) & 1], ((qa0 << shl) >> shr) & mk, ((qa1 << shl) >> shr) & mk,
                             ((qb0 << shl) >> shr) & mk, ((qb1 << shl) >> shr) & mk, ua, ub);
                }
            }
        }
    } else if (FMT == kBF16) {
        // bf16 weights times the token's bf16 hi and lo operands (family FB /
        // FBL), blocks 8 jj + (0..7) of 32; fragment order puts a lane's four
        // words of a row (k = 2t.., 8+2t.., 16+2t.., 24+2t..) together.  Only
        // lanes g = 0 supply the token (column 0 of B), so column 0 of D is the
        // row's dot product and the other columns stay zero.
        const uint32_t hb = tb + h.tx + jj * 512, lb = tb + h.ts + jj * 512;
        const bool own = g == 0;
#pragma unroll 2
        for (int b = 0; b < 8; ++b) {
            const uint4 Bh = lds128(own ? hb + 64 * b + 16 * t : zaddr);
            const uint4 Bl = lds128(own ? lb + 64 * b + 16 * t : zaddr);
            uint4 a[NR];
#pragma unroll
            for (int i = 0; i < NR; ++i) {
                const int r = rec_of(i) - jj * 32;
                a[i] = lds128(st + h.woff[0] + ((8 * jj + b) * 32 + r) * 64 + 16 * t);
            }
#pragma unroll
            for (int kc = 0; kc < 2; ++kc)
#pragma unroll
                for (int tl = 0; tl < NT; ++tl) {
                    const uint32_t a0 = sub4(a[2 * tl], 2 * kc), a1 = sub4(a[2 * tl + 1], 2 * kc);
                    const uint32_t a2 = sub4(a[2 * tl], 2 * kc + 1), a3 = sub4(a[2 * tl + 1], 2 * kc + 1);
                    mma16816_bf16(T.DD[tl][kc][0], a0, a1, a2, a3, sub4(Bh, 2 * kc), sub4(Bh, 2 * kc + 1));
                    mma16816_bf16(T.DD[tl][kc][1], a0, a1, a2, a3, sub4(Bl, 2 * kc), sub4(Bl, 2 * kc + 1));
                }
        }
    } else {   // Q8_0: blocks 8 jj + (0..7), pairs 8 half .. 8 half + 7, four accumulators per row tile
        uint4 cA[NR], cB[NR];   // rows: blocks t and t+4
#pragma unroll
        for (int i = 0; i < NR; ++i) {
            const int r = rec_of(i) - jj * 32;
            cA[i] = lds128(st + w1 + ((8 * jj + t) * 32 + r) * 32 + 16 * half);
            cB[i] = lds128(st + w1 + ((8 * jj + t + 4) * 32 + r) * 32 + 16 * half);
        }
        uint32_t XA[8], XB[8];
        ld_frag8(own0 ? xb + 64 * t + 32 * half : zaddr, XA);
        ld_frag8(own1 ? xb + 64 * (t + 4) + 32 * half : zaddr, XB);
#pragma unroll
        for (int mm = 0; mm < 8; ++mm) {
            const int wi = mm >> 1, sh = (mm & 1) ? 8 : 0, a = mm & 3;
#pragma unroll
            for (int tl = 0; tl < NT; ++tl)
                mma16816(T.DD[tl][a >> 1][a & 1], (sub4(cA[2 * tl], wi) >> sh) & 0x00FF00FFu,
                         (sub4(cA[2 * tl + 1], wi) >> sh) & 0x00FF00FFu, (sub4(cB[2 * tl], wi) >> sh) & 0x00FF00FFu,
                         (sub4(cB[2 * tl + 1], wi) >> sh) & 0x00FF00FFu, XA[mm], XB[mm]);
        }
    }
}

template <int FMT, int NT>
__device__ __forceinline__ void tile_epi(const Geo& h, uint32_t st, int jj, int half, int rt0, int tk,
                                         const TileAcc<NT>& T, float (&acc)[4]) {
    constexpr int NR = 2 * NT;
    const int lane = threadIdx.x & 31, g = lane >> 2, t = lane & 3;
    const int w0 = h.woff[0], w1 = h.woff[1], w2 = h.woff[2];
    const uint32_t tb = st + h.tok0 + tk * h.tstride;
    const uint32_t sb = tb + h.ts + jj * (kStatFloats * 4);
    const int rbase = jj * 32 + 16 * rt0 + g;
    auto rec_of = [&](int i) { return rbase + 16 * (i >> 1) + 8 * (i & 1); };

    if (FMT == kBF16) {
        // column 0 of D holds each row's sum (the other columns are zero)
#pragma unroll
        for (int i = 0; i < NR; ++i) {
            const int tl = i >> 1, hl = i & 1;
            acc[i] += (T.DD[tl][0][0][2 * hl] + T.DD[tl][0][1][2 * hl]) + (T.DD[tl][1][0][2 * hl] + T.DD[tl][1][1][2 * hl]);
        }
        return;
    }
    if (FMT == kQ2K || FMT == kQ3K || FMT == kQ6K) {
        // slot-ordered scale fields of each row: slot 4t + b (b = 2 * group + col)
        // holds the lane's sub-block of D[group][col].  Fields are turned into
        // fp16 pairs (b0, b2) / (b1, b3) whose values are field * 2^-24 (masked
        // bits in the mantissa of an fp16 subnormal), then widened to fp32; the
        // 2^24 is folded into d (d * 2^24 <= 2^40, exact).
        const float cf0 = ldsf(sb + 4 * (kStatC + t)), cf1 = ldsf(sb + 4 * (kStatC + 4 + t));
        const uint4 Su = lds128(sb + 4 * (kStatS16 + 4 * t));
        const float S[4] = {__uint_as_float(Su.x), __uint_as_float(Su.y), __uint_as_float(Su.z),
                            __uint_as_float(Su.w)};
        auto h2pair = [](uint32_t bits) { return __half22float2(*reinterpret_cast<const __half2*>(&bits)); };
#pragma unroll
        for (int i = 0; i < NR; ++i) {
            const int tl = i >> 1, hl = i & 1;
            float D[2][2];
#pragma unroll
            for (int gm = 0; gm < 2; ++gm)
#pragma unroll
                for (int cc = 0; cc < 2; ++cc)
                    D[gm][cc] = T.DD[tl][gm][0][2 * hl + cc] + T.DD[tl][gm][1][2 * hl + cc];
            const int rec = rec_of(i);
            const float d = h2f(lds16(st + w0 + rec * 2)) * 16777216.0f;
            if (FMT == kQ6K) {
                // scale bytes hold s + 128: masked into fp16 subnormal pairs
                // (s + 128) * 2^-24, minus 128 * 2^-24 (exact), widened; the
                // 2^24 is folded into d
                const uint32_t f = lds32(st + w1 + rec * 16 + 4 * t);
                const uint32_t fa = f & 0x00FF00FFu, fb = (f >> 8) & 0x00FF00FFu;
                const __half2 o128 = __halves2half2(__ushort_as_half((unsigned short)128), __ushort_as_half((unsigned short)128));
                const __half2 va = __hsub2(*reinterpret_cast<const __half2*>(&fa), o128);
                const __half2 vb = __hsub2(*reinterpret_cast<const __half2*>(&fb), o128);
                const float2 s02 = __half22float2(va), s13 = __half22float2(vb);   // slots (0, 2), (1, 3)
                const float P0 = fmaf(D[0][0], cf0, -32.0f * S[0]), P1 = fmaf(D[0][1], cf0, -32.0f * S[1]);
                const float P2 = fmaf(D[1][0], cf1, -32.0f * S[2]), P3 = fmaf(D[1][1], cf1, -32.0f * S[3]);
                const float a = fmaf(s13.y, P3, fmaf(s02.y, P2, fmaf(s13.x, P1, s02.x * P0)));
                acc[i] = fmaf(d, a, acc[i]);
            } else if (FMT == kQ2K) {
                // byte b = sc | m << 4; bytes 1 and 3 moved down to bytes 0 and 2
                const float dm = h2f(lds16(st + w1 + rec * 2)) * 1048576.0f;   // m sits 4 bits up: 2^-20
                const uint32_t f = lds32(st + w2 + rec * 16 + 4 * t);
                const uint32_t fo = __byte_perm(f, 0u, 0x7371u);
                const float2 s02 = h2pair(f & 0x000F000Fu), s13 = h2pair(fo & 0x000F000Fu);
                const float2 m02 = h2pair(f & 0x00F000F0u), m13 = h2pair(fo & 0x00F000F0u);
                const float a0 = fmaf(s13.x, D[0][1], s02.x * D[0][0]);
                const float a1 = fmaf(s13.y, D[1][1], s02.y * D[1][0]);
                const float am = fmaf(m13.y, S[3], fmaf(m02.y, S[2], fmaf(m13.x, S[1], m02.x * S[0])));
                acc[i] += fmaf(d, fmaf(cf1, a1, cf0 * a0), -dm * am);
            } else {
                // 6-bit scale s (stored s + 32): low nibble of slot u at bits 4u..4u+3
                // of bytes 0-7, high two bits at bits 2u..2u+1 of bytes 8-11
                const uint32_t sp = st + w1 + rec * 12;
                const uint32_t lo = lds16(sp + 2 * t), hi = lds8(sp + 8 + t);
                const uint32_t u = __byte_perm(lo, 0u, 0x7170u);   // halves: n0 | n1 << 4, n2 | n3 << 4
                const uint32_t v = __byte_perm(hi, 0u, 0x7070u);   // both halves: h0 | h1 << 2 | h2 << 4 | h3 << 6
                // (n0 + 16 h0, n2 + 16 h2) and (n1 + 16 h1, n3 + 16 h3), exact in fp16
                // subnormals (the 2-bit fields weighed up to bit 4 by the multipliers),
                // then minus 32
                const __half2 c32 = __halves2half2(__ushort_as_half((unsigned short)32), __ushort_as_half((unsigned short)32));
                const uint32_t uA = u & 0x000F000Fu, uB = (u >> 4) & 0x000F000Fu;
                const __half2 lA = *reinterpret_cast<const __half2*>(&uA);
                const __half2 lB = *reinterpret_cast<const __half2*>(&uB);
                const uint32_t hA = v & 0x00300003u, hB = v & 0x00C0000Cu;
                const __half2 mA = __halves2half2(__float2half(16.0f), __float2half(1.0f));
                const __half2 mB = __halves2half2(__float2half(4.0f), __float2half(0.25f));
                const __half2 sA = __hsub2(__hfma2(*reinterpret_cast<const __half2*>(&hA), mA, lA), c32);
                const __half2 sB = __hsub2(__hfma2(*reinterpret_cast<const __half2*>(&hB), mB, lB), c32);
                const float2 vA = __half22float2(sA), vB = __half22float2(sB);   // slots (0, 2), (1, 3)
                const float P0 = fmaf(D[0][0], cf0, -4.0f * S[0]), P1 = fmaf(D[0][1], cf0, -4.0f * S[1]);
                const float P2 = fmaf(D[1][0], cf1, -4.0f * S[2]), P3 = fmaf(D[1][1], cf1, -4.0f * S[3]);
                const float a = fmaf(vB.y, P3, fmaf(vA.y, P2, fmaf(vB.x, P1, vA.x * P0)));
                acc[i] = fmaf(d, a, acc[i]);
            }
        }
    } else if (FMT == kQ4K) {
        const uint2 Cu = lds64(sb + 4 * (kStatC + 2 * t)), Su = lds64(sb + 4 * (kStatS32 + 2 * t));
        const float cf0 = __uint_as_float(Cu.x), cf1 = __uint_as_float(Cu.y);
        const float S0 = __uint_as_float(Su.x), S1 = __uint_as_float(Su.y);
#pragma unroll
        for (int i = 0; i < NR; ++i) {
            const int tl = i >> 1, hl = i & 1, rec = rec_of(i);
            const float d = h2f(lds16(st + w0 + rec * 2));
            const float dm = h2f(lds16(st + w1 + rec * 2));
            const uint32_t sp = st + w2 + rec * 12;
            const uint32_t f = lds16(sp + 2 * t), hi = lds8(sp + 8 + t);
            const float sc0 = (float)((f & 15u) | ((hi & 3u) << 4));
            const float m0 = (float)(((f >> 4) & 15u) | (((hi >> 2) & 3u) << 4));
            const float sc1 = (float)(((f >> 8) & 15u) | (((hi >> 4) & 3u) << 4));
            const float m1 = (float)(((f >> 12) & 15u) | (((hi >> 6) & 3u) << 4));
            const float D0 = (T.DD[tl][0][0][2 * hl] + T.DD[tl][0][1][2 * hl]) + (T.DD[tl][1][0][2 * hl] + T.DD[tl][1][1][2 * hl]);
            const float D1 = (T.DD[tl][0][0][2 * hl + 1] + T.DD[tl][0][1][2 * hl + 1]) +
                             (T.DD[tl][1][0][2 * hl + 1] + T.DD[tl][1][1][2 * hl + 1]);
            const float a_sc = fmaf(sc1 * cf1, D1, sc0 * cf0 * D0);
            const float a_m = fmaf(m1, S1, m0 * S0);
            acc[i] += fmaf(d, a_sc, -dm * a_m);
        }
    } else {
        const uint2 Cu = lds64(sb + 4 * (kStatC + 2 * t)), Su = lds64(sb + 4 * (kStatS32 + 2 * t));
        const float cf0 = __uint_as_float(Cu.x), cf1 = __uint_as_float(Cu.y);
        // codes are stored q + 128: one half removes 128 * sum(x) per block
        const float o0 = half ? 0.0f : 128.0f * __uint_as_float(Su.x);
        const float o1 = half ? 0.0f : 128.0f * __uint_as_float(Su.y);
#pragma unroll
        for (int i = 0; i < NR; ++i) {
            const int tl = i >> 1, hl = i & 1, r = rec_of(i) - jj * 32;
            const float d0 = h2f(lds16(st + w0 + ((8 * jj + 2 * t) * 32 + r) * 2));
            const float d1 = h2f(lds16(st + w0 + ((8 * jj + 2 * t + 1) * 32 + r) * 2));
            const float D0 = (T.DD[tl][0][0][2 * hl] + T.DD[tl][0][1][2 * hl]) + (T.DD[tl][1][0][2 * hl] + T.DD[tl][1][1][2 * hl]);
            const float D1 = (T.DD[tl][0][0][2 * hl + 1] + T.DD[tl][0][1][2 * hl + 1]) +
                             (T.DD[tl][1][0][2 * hl + 1] + T.DD[tl][1][1][2 * hl + 1]);
            acc[i] += fmaf(d1, fmaf(D1, cf1, -o1), d0 * fmaf(D0, cf0, -o0));
        }
    }
}

// Two tokens of a multi-token item through one 16-row tile (rows 16 rt + g,
// + 8) of a Q2_K superblock.  The masked code operands do not depend on the
// token, so each is built once for both tokens' MMAs, and the epilogue's
// scale conversions are shared; per token the arithmetic is that of
// tile_mma<kQ2K, 1> and tile_epi<kQ2K, 1> in the same order, so the sums are
// the ones the per-token passes give.  acc[k][hl]: token tk0 + k's sum of
// row 16 rt + g + 8 hl, updated in place.
__device__ __forceinline__ void tile_pair_q2k(const Geo& h, uint32_t st, int jj, int rt, int tk0, uint32_t zaddr,
                                              float (&acc)[2][2]) {
    const int lane = threadIdx.x & 31, g = lane >> 2, t = lane & 3;
    const bool own0 = g == t, own1 = g == t + 4;
    const int w0 = h.woff[0], w1 = h.woff[1], w2 = h.woff[2], w3 = h.woff[3];
    const uint32_t tbA = st + h.tok0 + tk0 * h.tstride, tbB = tbA + h.tstride;
    const uint32_t xbA = tbA + h.tx + jj * 512, xbB = tbB + h.tx + jj * 512;
    const int rbase = jj * 32 + 16 * rt + g;
    const uint4 c0 = lds128(st + w3 + rbase * 64 + 16 * t), c1 = lds128(st + w3 + (rbase + 8) * 64 + 16 * t);
    float D[2][2][2][4];   // [token][sub-block group][pair parity][D fragment]
#pragma unroll
    for (int i = 0; i < 32; ++i) (&D[0][0][0][0])[i] = 0.0f;
#pragma unroll
    for (int gm = 0; gm < 2; ++gm) {
        uint32_t XA0[8], XB0[8], XA1[8], XB1[8];
        ld_frag8(own0 ? xbA + 32 * (8 * gm + t) : zaddr, XA0);
        ld_frag8(own1 ? xbA + 32 * (8 * gm + 4 + t) : zaddr, XB0);
        ld_frag8(own0 ? xbB + 32 * (8 * gm + t) : zaddr, XA1);
        ld_frag8(own1 ? xbB + 32 * (8 * gm + 4 + t) : zaddr, XB1);
        const uint32_t qa0 = sub4(c0, 2 * gm), qa1 = sub4(c1, 2 * gm);
        const uint32_t qb0 = sub4(c0, 2 * gm + 1), qb1 = sub4(c1, 2 * gm + 1);
        const uint32_t sa0 = qa0 >> 10, sa1 = qa1 >> 10, sb0 = qb0 >> 10, sb1 = qb1 >> 10;
#pragma unroll
        for (int m = 0; m < 8; ++m) {
            const uint32_t mk = 0x00030003u << (m <= 4 ? 2 * m : 2 * (m - 5));
            const bool sh = m > 4;
            const uint32_t a0 = (sh ? sa0 : qa0) & mk, a1 = (sh ? sa1 : qa1) & mk;
            const uint32_t a2 = (sh ? sb0 : qb0) & mk, a3 = (sh ? sb1 : qb1) & mk;
            mma16816(D[0][gm][m & 1], a0, a1, a2, a3, XA0[m], XB0[m]);
            mma16816(D[1][gm][m & 1], a0, a1, a2, a3, XA1[m], XB1[m]);
        }
    }
    auto h2pair = [](uint32_t bits) { return __half22float2(*reinterpret_cast<const __half2*>(&bits)); };
    float cf0[2], cf1[2], S[2][4];
#pragma unroll
    for (int k = 0; k < 2; ++k) {
        const uint32_t sb = (k ? tbB : tbA) + h.ts + jj * (kStatFloats * 4);
        cf0[k] = ldsf(sb + 4 * (kStatC + t)); cf1[k] = ldsf(sb + 4 * (kStatC + 4 + t));
        const uint4 Su = lds128(sb + 4 * (kStatS16 + 4 * t));
        S[k][0] = __uint_as_float(Su.x); S[k][1] = __uint_as_float(Su.y);
        S[k][2] = __uint_as_float(Su.z); S[k][3] = __uint_as_float(Su.w);
    }
#pragma unroll
    for (int hl = 0; hl < 2; ++hl) {
        const int rec = rbase + 8 * hl;
        const float d = h2f(lds16(st + w0 + rec * 2)) * 16777216.0f;
        const float dm = h2f(lds16(st + w1 + rec * 2)) * 1048576.0f;   // m sits 4 bits up: 2^-20
        const uint32_t f = lds32(st + w2 + rec * 16 + 4 * t);
        const uint32_t fo = __byte_perm(f, 0u, 0x7371u);
        const float2 s02 = h2pair(f & 0x000F000Fu), s13 = h2pair(fo & 0x000F000Fu);
        const float2 m02 = h2pair(f & 0x00F000F0u), m13 = h2pair(fo & 0x00F000F0u);
#pragma unroll
        for (int k = 0; k < 2; ++k) {
            float Dk[2][2];
#pragma unroll
            for (int gm = 0; gm < 2; ++gm)
#pragma unroll
                for (int cc = 0; cc < 2; ++cc) Dk[gm][cc] = D[k][gm][0][2 * hl + cc] + D[k][gm][1][2 * hl + cc];
            const float a0 = fmaf(s13.x, Dk[0][1], s02.x * Dk[0][0]);
            const float a1 = fmaf(s13.y, Dk[1][1], s02.y * Dk[1][0]);
            const float am = fmaf(m13.y, S[k][3], fmaf(m02.y, S[k][2], fmaf(m13.x, S[k][1], m02.x * S[k][0])));
            const float v = fmaf(d, fmaf(cf1[k], a1, cf0[k] * a0), -dm * am);
            acc[k][hl] += v;
        }
    }
}

// Q3_K, as tile_pair_q2k: code q = low2 + 4 hbit, the low bits through the
// Q2_K MMAs, the high bits through MMAs of their own against the token's
// operand scaled by 4 * 2^(pos(m) - m) (as tile_mma<kQ3K, 1>); the 6-bit
// scales (stored + 32) are widened once for both tokens (as tile_epi).
__device__ __forceinline__ void tile_pair_q3k(const Geo& h, uint32_t st, int jj, int rt, int tk0, uint32_t zaddr,
                                              float (&acc)[2][2]) {
    const int lane = threadIdx.x & 31, g = lane >> 2, t = lane & 3;
    const bool own0 = g == t, own1 = g == t + 4;
    const int w0 = h.woff[0], w1 = h.woff[1], w2 = h.woff[2], w3 = h.woff[3];
    const uint32_t tbA = st + h.tok0 + tk0 * h.tstride, tbB = tbA + h.tstride;
    const uint32_t xbA = tbA + h.tx + jj * 512, xbB = tbB + h.tx + jj * 512;
    const int rbase = jj * 32 + 16 * rt + g;
    const uint4 c0 = lds128(st + w2 + rbase * 64 + 16 * t), c1 = lds128(st + w2 + (rbase + 8) * 64 + 16 * t);
    const uint2 hv0 = lds64(st + w3 + rbase * 32 + 8 * t), hv1 = lds64(st + w3 + (rbase + 8) * 32 + 8 * t);
    float D[2][2][2][4];   // [token][sub-block group][pair parity][D fragment]
#pragma unroll
    for (int i = 0; i < 32; ++i) (&D[0][0][0][0])[i] = 0.0f;
    // one sub-block group at a time (each accumulator sees its MMAs in the
    // order of tile_mma<kQ3K, 1>: the low-bit pairs, then the high bits)
#pragma unroll
    for (int gm = 0; gm < 2; ++gm) {
        uint32_t XA[2][8], XB[2][8];   // [token][pair]
        ld_frag8(own0 ? xbA + 32 * (8 * gm + t) : zaddr, XA[0]);
        ld_frag8(own1 ? xbA + 32 * (8 * gm + 4 + t) : zaddr, XB[0]);
        ld_frag8(own0 ? xbB + 32 * (8 * gm + t) : zaddr, XA[1]);
        ld_frag8(own1 ? xbB + 32 * (8 * gm + 4 + t) : zaddr, XB[1]);
        const uint32_t qa0 = sub4(c0, 2 * gm), qa1 = sub4(c1, 2 * gm);
        const uint32_t qb0 = sub4(c0, 2 * gm + 1), qb1 = sub4(c1, 2 * gm + 1);
        const uint32_t sa0 = qa0 >> 10, sa1 = qa1 >> 10, sb0 = qb0 >> 10, sb1 = qb1 >> 10;
#pragma unroll
        for (int m = 0; m < 8; ++m) {
            const uint32_t mk = 0x00030003u << (m <= 4 ? 2 * m : 2 * (m - 5));
            const bool sh = m > 4;
            const uint32_t a0 = (sh ? sa0 : qa0) & mk, a1 = (sh ? sa1 : qa1) & mk;
            const uint32_t a2 = (sh ? sb0 : qb0) & mk, a3 = (sh ? sb1 : qb1) & mk;
            mma16816(D[0][gm][m & 1], a0, a1, a2, a3, XA[0][m], XB[0][m]);
            mma16816(D[1][gm][m & 1], a0, a1, a2, a3, XA[1][m], XB[1][m]);
        }
        const uint32_t ha0 = gm ? hv0.y : hv0.x, ha1 = gm ? hv1.y : hv1.x;
        const uint32_t hb0 = ha0 >> 8, hb1 = ha1 >> 8;
#pragma unroll
        for (int m = 0; m < 8; ++m) {
            const uint32_t mh = 0x00010001u << m;
            const int e = m <= 4 ? m + 2 : m - 8;
            const uint32_t sc16 = (uint32_t)(15 + e) << 10;
            const __half2 scl = __halves2half2(__ushort_as_half((unsigned short)sc16), __ushort_as_half((unsigned short)sc16));
            const uint32_t a0 = ha0 & mh, a1 = ha1 & mh, a2 = hb0 & mh, a3 = hb1 & mh;
#pragma unroll
            for (int k = 0; k < 2; ++k) {
                const __half2 xa = __hmul2(*reinterpret_cast<const __half2*>(&XA[k][m]), scl);
                const __half2 xb2 = __hmul2(*reinterpret_cast<const __half2*>(&XB[k][m]), scl);
                mma16816(D[k][gm][(m + 1) & 1], a0, a1, a2, a3, *reinterpret_cast<const uint32_t*>(&xa),
                         *reinterpret_cast<const uint32_t*>(&xb2));
            }
        }
    }
    float cf0[2], cf1[2], S[2][4];
#pragma unroll
    for (int k = 0; k < 2; ++k) {
        const uint32_t sb = (k ? tbB : tbA) + h.ts + jj * (kStatFloats * 4);
        cf0[k] = ldsf(sb + 4 * (kStatC + t)); cf1[k] = ldsf(sb + 4 * (kStatC + 4 + t));
        const uint4 Su = lds128(sb + 4 * (kStatS16 + 4 * t));
        S[k][0] = __uint_as_float(Su.x); S[k][1] = __uint_as_float(Su.y);
        S[k][2] = __uint_as_float(Su.z); S[k][3] = __uint_as_float(Su.w);
    }
#pragma unroll
    for (int hl = 0; hl < 2; ++hl) {
        const int rec = rbase + 8 * hl;
        const float d = h2f(lds16(st + w0 + rec * 2)) * 16777216.0f;
        const uint32_t sp = st + w1 + rec * 12;
        const uint32_t lo = lds16(sp + 2 * t), hi = lds8(sp + 8 + t);
        const uint32_t u = __byte_perm(lo, 0u, 0x7170u);
        const uint32_t v = __byte_perm(hi, 0u, 0x7070u);
        const __half2 c32 = __halves2half2(__ushort_as_half((unsigned short)32), __ushort_as_half((unsigned short)32));
        const uint32_t uA = u & 0x000F000Fu, uB = (u >> 4) & 0x000F000Fu;
        const __half2 lA = *reinterpret_cast<const __half2*>(&uA);
        const __half2 lB = *reinterpret_cast<const __half2*>(&uB);
        const uint32_t hA = v & 0x00300003u, hB = v & 0x00C0000Cu;
        const __half2 mA = __halves2half2(__float2half(16.0f), __float2half(1.0f));
        const __half2 mB = __halves2half2(__float2half(4.0f), __float2half(0.25f));
        const __half2 sA = __hsub2(__hfma2(*reinterpret_cast<const __half2*>(&hA), mA, lA), c32);
        const __half2 sB = __hsub2(__hfma2(*reinterpret_cast<const __half2*>(&hB), mB, lB), c32);
        const float2 vA = __half22float2(sA), vB = __half22float2(sB);
#pragma unroll
        for (int k = 0; k < 2; ++k) {
            float Dk[2][2];
#pragma unroll
            for (int gm = 0; gm < 2; ++gm)
#pragma unroll
                for (int cc = 0; cc < 2; ++cc) Dk[gm][cc] = D[k][gm][0][2 * hl + cc] + D[k][gm][1][2 * hl + cc];
            const float P0 = fmaf(Dk[0][0], cf0[k], -4.0f * S[k][0]), P1 = fmaf(Dk[0][1], cf0[k], -4.0f * S[k][1]);
            const float P2 = fmaf(Dk[1][0], cf1[k], -4.0f * S[k][2]), P3 = fmaf(Dk[1][1], cf1[k], -4.0f * S[k][3]);
            const float a = fmaf(vB.y, P3, fmaf(vA.y, P2, fmaf(vB.x, P1, vA.x * P0)));
            acc[k][hl] = fmaf(d, a, acc[k][hl]);
        }
    }
}

// Q4_K, as tile_pair_q2k (tile_mma<kQ4K, 1> and tile_epi<kQ4K, 1> per token).
__device__ __forceinline__ void tile_pair_q4k(const Geo& h, uint32_t st, int jj, int rt, int tk0, uint32_t zaddr,
                                              float (&acc)[2][2]) {
    const int lane = threadIdx.x & 31, g = lane >> 2, t = lane & 3;
    const bool own0 = g == t, own1 = g == t + 4;
    const int w0 = h.woff[0], w1 = h.woff[1], w2 = h.woff[2], w3 = h.woff[3];
    const uint32_t tbA = st + h.tok0 + tk0 * h.tstride, tbB = tbA + h.tstride;
    const uint32_t xbA = tbA + h.tx + jj * 512, xbB = tbB + h.tx + jj * 512;
    const int rbase = jj * 32 + 16 * rt + g;
    const int r0 = rbase - jj * 32, r1 = r0 + 8;
    const uint4 cA0 = lds128(st + w3 + ((jj * 2 + 0) * 32 + r0) * 64 + 16 * t);
    const uint4 cA1 = lds128(st + w3 + ((jj * 2 + 0) * 32 + r1) * 64 + 16 * t);
    const uint4 cB0 = lds128(st + w3 + ((jj * 2 + 1) * 32 + r0) * 64 + 16 * t);
    const uint4 cB1 = lds128(st + w3 + ((jj * 2 + 1) * 32 + r1) * 64 + 16 * t);
    float D[2][2][2][4];
#pragma unroll
    for (int i = 0; i < 32; ++i) (&D[0][0][0][0])[i] = 0.0f;
    // one half of the pairs at a time (accumulator D[.][hm][.] takes only hm's)
#pragma unroll
    for (int hm = 0; hm < 2; ++hm) {
        uint32_t XA[2][8], XB[2][8];   // [token][pair]
        ld_frag8(own0 ? xbA + 64 * t + 32 * hm : zaddr, XA[0]);
        ld_frag8(own1 ? xbA + 64 * (t + 4) + 32 * hm : zaddr, XB[0]);
        ld_frag8(own0 ? xbB + 64 * t + 32 * hm : zaddr, XA[1]);
        ld_frag8(own1 ? xbB + 64 * (t + 4) + 32 * hm : zaddr, XB[1]);
#pragma unroll
        for (int mm = 0; mm < 8; ++mm) {
            const int m = 8 * hm + mm, wi = m >> 2, j = m & 3;
            const uint32_t mk = (j & 1) ? 0x00F000F0u : 0x000F000Fu;
            const int sh = j < 2 ? 0 : 8;
            const uint32_t a0 = (sub4(cA0, wi) >> sh) & mk, a1 = (sub4(cA1, wi) >> sh) & mk;
            const uint32_t a2 = (sub4(cB0, wi) >> sh) & mk, a3 = (sub4(cB1, wi) >> sh) & mk;
            mma16816(D[0][hm][mm & 1], a0, a1, a2, a3, XA[0][mm], XB[0][mm]);
            mma16816(D[1][hm][mm & 1], a0, a1, a2, a3, XA[1][mm], XB[1][mm]);
        }
    }
    float cf0[2], cf1[2], S0[2], S1[2];
#pragma unroll
    for (int k = 0; k < 2; ++k) {
        const uint32_t sb = (k ? tbB : tbA) + h.ts + jj * (kStatFloats * 4);
        const uint2 Cu = lds64(sb + 4 * (kStatC + 2 * t)), Su = lds64(sb + 4 * (kStatS32 + 2 * t));
        cf0[k] = __uint_as_float(Cu.x); cf1[k] = __uint_as_float(Cu.y);
        S0[k] = __uint_as_float(Su.x); S1[k] = __uint_as_float(Su.y);
    }
#pragma unroll
    for (int hl = 0; hl < 2; ++hl) {
        const int rec = rbase + 8 * hl;
        const float d = h2f(lds16(st + w0 + rec * 2));
        const float dm = h2f(lds16(st + w1 + rec * 2));
        const uint32_t sp = st + w2 + rec * 12;
        const uint32_t f = lds16(sp + 2 * t), hi = lds8(sp + 8 + t);
        const float sc0 = (float)((f & 15u) | ((hi & 3u) << 4));
        const float m0 = (float)(((f >> 4) & 15u) | (((hi >> 2) & 3u) << 4));
        const float sc1 = (float)(((f >> 8) & 15u) | (((hi >> 4) & 3u) << 4));
        const float m1 = (float)(((f >> 12) & 15u) | (((hi >> 6) & 3u) << 4));
#pragma unroll
        for (int k = 0; k < 2; ++k) {
            const float D0 = (D[k][0][0][2 * hl] + D[k][0][1][2 * hl]) + (D[k][1][0][2 * hl] + D[k][1][1][2 * hl]);
            const float D1 = (D[k][0][0][2 * hl + 1] + D[k][0][1][2 * hl + 1]) +
                             (D[k][1][0][2 * hl + 1] + D[k][1][1][2 * hl + 1]);
            const float a_sc = fmaf(sc1 * cf1[k], D1, sc0 * cf0[k] * D0);
            const float a_m = fmaf(m1, S1[k], m0 * S0[k]);
            const float v = fmaf(d, a_sc, -dm * a_m);
            acc[k][hl] += v;
        }
    }
}

// Q8_0, as tile_pair_q2k: one half of each superblock's code pairs
// (tile_mma<kQ80, 1> and tile_epi<kQ80, 1> per token).
__device__ __forceinline__ void tile_pair_q80(const Geo& h, uint32_t st, int jj, int half, int rt, int tk0,
                                              uint32_t zaddr, float (&acc)[2][2]) {
    const int lane = threadIdx.x & 31, g = lane >> 2, t = lane & 3;
    const bool own0 = g == t, own1 = g == t + 4;
    const int w0 = h.woff[0], w1 = h.woff[1];
    const uint32_t tbA = st + h.tok0 + tk0 * h.tstride, tbB = tbA + h.tstride;
    const uint32_t xbA = tbA + h.tx + jj * 512, xbB = tbB + h.tx + jj * 512;
    const int rbase = jj * 32 + 16 * rt + g;
    const int r0 = rbase - jj * 32, r1 = r0 + 8;
    const uint4 cA0 = lds128(st + w1 + ((8 * jj + t) * 32 + r0) * 32 + 16 * half);
    const uint4 cA1 = lds128(st + w1 + ((8 * jj + t) * 32 + r1) * 32 + 16 * half);
    const uint4 cB0 = lds128(st + w1 + ((8 * jj + t + 4) * 32 + r0) * 32 + 16 * half);
    const uint4 cB1 = lds128(st + w1 + ((8 * jj + t + 4) * 32 + r1) * 32 + 16 * half);
    float D[2][2][2][4];
#pragma unroll
    for (int i = 0; i < 32; ++i) (&D[0][0][0][0])[i] = 0.0f;
    uint32_t XA[2][8], XB[2][8];   // [token][pair]
    ld_frag8(own0 ? xbA + 64 * t + 32 * half : zaddr, XA[0]);
    ld_frag8(own1 ? xbA + 64 * (t + 4) + 32 * half : zaddr, XB[0]);
    ld_frag8(own0 ? xbB + 64 * t + 32 * half : zaddr, XA[1]);
    ld_frag8(own1 ? xbB + 64 * (t + 4) + 32 * half : zaddr, XB[1]);
#pragma unroll
    for (int mm = 0; mm < 8; ++mm) {
        const int wi = mm >> 1, sh = (mm & 1) ? 8 : 0, a = mm & 3;
        const uint32_t a0 = (sub4(cA0, wi) >> sh) & 0x00FF00FFu, a1 = (sub4(cA1, wi) >> sh) & 0x00FF00FFu;
        const uint32_t a2 = (sub4(cB0, wi) >> sh) & 0x00FF00FFu, a3 = (sub4(cB1, wi) >> sh) & 0x00FF00FFu;
        mma16816(D[0][a >> 1][a & 1], a0, a1, a2, a3, XA[0][mm], XB[0][mm]);
        mma16816(D[1][a >> 1][a & 1], a0, a1, a2, a3, XA[1][mm], XB[1][mm]);
    }
    float cf0[2], cf1[2], o0[2], o1[2];
#pragma unroll
    for (int k = 0; k < 2; ++k) {
        const uint32_t sb = (k ? tbB : tbA) + h.ts + jj * (kStatFloats * 4);
        const uint2 Cu = lds64(sb + 4 * (kStatC + 2 * t)), Su = lds64(sb + 4 * (kStatS32 + 2 * t));
        cf0[k] = __uint_as_float(Cu.x); cf1[k] = __uint_as_float(Cu.y);
        o0[k] = half ? 0.0f : 128.0f * __uint_as_float(Su.x);
        o1[k] = half ? 0.0f : 128.0f * __uint_as_float(Su.y);
    }
#pragma unroll
    for (int hl = 0; hl < 2; ++hl) {
        const int r = (rbase + 8 * hl) - jj * 32;
        const float d0 = h2f(lds16(st + w0 + ((8 * jj + 2 * t) * 32 + r) * 2));
        const float d1 = h2f(lds16(st + w0 + ((8 * jj + 2 * t + 1) * 32 + r) * 2));
#pragma unroll
        for (int k = 0; k < 2; ++k) {
            const float D0 = (D[k][0][0][2 * hl] + D[k][0][1][2 * hl]) + (D[k][1][0][2 * hl] + D[k][1][1][2 * hl]);
            const float D1 = (D[k][0][0][2 * hl + 1] + D[k][0][1][2 * hl + 1]) +
                             (D[k][1][0][2 * hl + 1] + D[k][1][1][2 * hl + 1]);
            const float v = fmaf(d1, fmaf(D1, cf1[k], -o1[k]), d0 * fmaf(D0, cf0[k], -o0[k]));
            acc[k][hl] += v;
        }
    }
}

// The warp's superblocks col, col + kCols, ... of a stage, one tile at a time.
template <int FMT>
__device__ __forceinline__ void tile_cols(const Geo& h, uint32_t st, int col, int ks, int rt0, int tk,
                                          uint32_t zaddr, float (&acc)[4]) {
    for (int jj = col; jj < ks; jj += kCols) {
        TileAcc<kNT> T0;
        tile_mma<FMT, kNT>(h, st, jj, 0, rt0, tk, zaddr, T0);
        tile_epi<FMT, kNT>(h, st, jj, 0, rt0, tk, T0, acc);
    }
}


// MT: most tokens an item of this launch carries (1 when the call has one token)
template <int MT>
__global__ void __launch_bounds__(kThreads, 1) ffn_kernel(const __grid_constant__ ExpertTab tab,
                                                          const __grid_constant__ DecodeArgs A) {
    extern __shared__ __align__(128) uint8_t smem[];
    constexpr int kRedBufs = 2;                         // item-end reduction buffers
    __shared__ SlotCache sc;
    __shared__ int32_t s_perm[kMaxCachedAssign];
    __shared__ float s_wts[kMaxCachedAssign];   // routing weights by assignment (the first kMaxCachedAssign)
    __shared__ __align__(8) uint64_t bars[2 * kNST];
    __shared__ Hdr hdr[kNST];
    __shared__ float red[kRedBufs][kConsumers][2][MT][32];
    __shared__ int s_posted[kNST];   // last stage index posted to each ring slot
    __shared__ int s_fail;           // a bounded wait ran out somewhere in the CTA
    __shared__ int s_touch;
    __shared__ __align__(16) uint32_t zero_blk[8];   // operand B of the lanes that supply none
    __shared__ Geo geo[2][kNumFormats][kDecodeTok];
    const Dims& d = A.d;
    // ---- set-up that does not depend on the routing result runs before the
    // wait for the previous kernel (overlapping its tail)
    {
        // stage geometry (host-computed) into shared memory, one word per thread
        static_assert(sizeof(geo) % 4 == 0, "geometry table");
        const uint32_t* src = reinterpret_cast<const uint32_t*>(&A.geo[0][0][0]);
        uint32_t* dst = reinterpret_cast<uint32_t*>(&geo[0][0][0]);
        for (int i = threadIdx.x; i < (int)(sizeof(geo) / 4); i += kThreads) dst[i] = src[i];
    }
    const uint32_t bar0 = (uint32_t)__cvta_generic_to_shared(bars);
    if (threadIdx.x < kNST) s_posted[threadIdx.x] = -1;
    if (threadIdx.x < 8) zero_blk[threadIdx.x] = 0u;
    if (threadIdx.x == 0) s_fail = 0;
    {
        // Touch the expert table (a kernel parameter) once on this SM, so the
        // slot table's lookups made when the routing result arrives hit the
        // constant cache.
        uintptr_t v = 0;
        for (int i = threadIdx.x; i < 3 * (d.E + 1); i += kThreads) v |= reinterpret_cast<uintptr_t>(tab.p[i / 3][i % 3]);
        for (int i = threadIdx.x; i < d.E + 1; i += kThreads) v |= (uintptr_t)tab.fmt[i][0] << 8;
        if (v == 1) s_touch = 1;   // never true (pointers are 256-byte aligned); keeps the loads
    }
    const uint32_t zaddr = (uint32_t)__cvta_generic_to_shared(zero_blk);
    if (threadIdx.x == 0) {
        for (int s = 0; s < kNST; ++s) {
            mbar_init(bar0 + 8 * s, 1);                       // full[s]: producer arrival + tx bytes
            mbar_init(bar0 + 8 * (kNST + s), kConsumers);     // empty[s]: one arrival per consumer warp
        }
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    }
    // The shared expert's gate/up items (item ids 0 .. n_sh_items - 1) need no
    // routing result: its slot is known from the shapes, so they start before
    // the wait for the routing kernel.  (The tokens' prepared activations come
    // from the logits kernel, which completed before the routing kernel let
    // this grid launch.)
    const int n_sh_blocks = d.has_shared ? (d.I / 32) * ((d.T + kDecodeTok - 1) / kDecodeTok) : 0;
    const int n_sh_items = A.split_shared ? 2 * n_sh_blocks : n_sh_blocks;
    if (threadIdx.x == 0 && n_sh_items > 0) {
        sc.pre_gu[0] = 0; sc.pre_gu[1] = n_sh_items;
        sc.e[0] = d.E; sc.first[0] = 0; sc.ntot[0] = d.T;
    }
    if (threadIdx.x < 3 && d.has_shared) {
        sc.p[0][threadIdx.x] = tab.p[d.E][threadIdx.x];
        sc.fmt[0][threadIdx.x] = tab.fmt[d.E][threadIdx.x];
    }
    __syncthreads();
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const uint32_t ring = (uint32_t)__cvta_generic_to_shared(smem);

    if (warp == kProducerWarp) {
        // ===================== producer (dedicated warp) =====================
        // The CTA claims items from the per-call counter.  Per phase (one
        // tensor, or one 32-row block of down, of one item) every lane owns at
        // most one copy: lanes 0..3 a weight plane, lanes 4.. one piece of one
        // token (family fragments or statistics).  A stage then only advances
        // the source by the stage's first superblock.
        const VecSrc vx{A.xq, A.xs, (size_t)kFamSlots * A.nsbx * 256, (size_t)A.nsbx * kStatFloats, A.nsbx};
        const VecSrc vh{A.hq, A.hs, (size_t)kFamSlots * A.nsbi * 256, (size_t)A.nsbi * kStatFloats, A.nsbi};
        int cur_gu = 0, cur_dn = 0, p_q = 0;
        // weights are read once per call: evict-first in L2, so they do not
        // displace the activations, h and partial outputs the kernel shares
        const uint64_t wpol = evict_first_policy();
        ItemDesc P;
        int fmt0 = 1, fmt1 = 1;
        // the routing result: slot table (one level of independent loads; the
        // plan holds each slot's expert, first entry and token count) and the
        // cached permutation
        int n_slots = n_sh_items > 0 ? 1 : 0, n_gu = n_sh_items, n_items = n_sh_items;
        bool routed = false;
        // bounded acquire-spin on a word another kernel publishes with release
        auto wait_word = [&](const uint32_t* wp, uint32_t target) {
            if (lane == 0 && ld_acquire(wp) < target) {
                const uint64_t t0 = global_ns();
                // polled with a back-off: every CTA's producer polls the same word
                while (ld_acquire(wp) < target) {
                    if (global_ns() - t0 > A.wait_ns) { atomicOr(A.err, kErrReady); s_fail = 1; break; }
                    __nanosleep(256);
                }
            }
            __syncwarp();
            (void)ld_acquire(wp);   // every lane acquires before its own reads and copies
            asm volatile("fence.proxy.async.global;" ::: "memory");
        };
        bool tokens_in = false;   // the logits kernel's prepared tokens are written
        auto wait_routing = [&]() {
            // the routing result: published by the last CTA of the logits kernel
            wait_word(A.route_ready, 1u);
            tokens_in = true;   // published after every logits CTA counted itself
            // read through L2 (ld.global.cg): an SM's L1 may still hold lines
            // of an earlier call
            // The slot count and the first 32 slots' entries (every slot of a
            // call with at most 31 active experts) and the first 128 routed
            // entries of the permutation go out as one batch of independent
            // loads (one round trip); later passes only for larger calls.
            const int n_routed = min(d.T * d.K, kMaxCachedAssign);
            const int ns0 = __ldcg(&A.plan->n_slots);
            int pg0 = __ldcg(&A.plan->pre_gu[lane]), pd0 = __ldcg(&A.plan->pre_dn[lane]);
            int e0 = __ldcg(&A.plan->slot_e[lane]), f0 = __ldcg(&A.plan->slot_first[lane]);
            int nt0 = __ldcg(&A.plan->slot_ntot[lane]);
            int pv0[4];
            float wv0[4];
#pragma unroll
            for (int u = 0; u < 4; ++u) {
                const int i = 32 * u + lane;
                pv0[u] = i < n_routed ? __ldcg(A.perm + i) : 0;
                wv0[u] = i < n_routed ? __ldcg(A.wts + i) : 0.0f;
            }
            n_slots = ns0;
            for (int i = lane; i <= n_slots; i += 32) {
                int pg = pg0, pd = pd0, e = e0, first = f0, ntot = nt0;
                if (i >= 32) {
                    pg = __ldcg(&A.plan->pre_gu[i]); pd = __ldcg(&A.plan->pre_dn[i]);
                    if (i < n_slots) {
                        e = __ldcg(&A.plan->slot_e[i]);
                        first = __ldcg(&A.plan->slot_first[i]);
                        ntot = __ldcg(&A.plan->slot_ntot[i]);
                    }
                }
                // the plan counts one gate/up item per shared block; with the K
                // split the shared slot has two
                sc.pre_gu[i] = pg + (i >= 1 && A.split_shared ? n_sh_blocks : 0);
                sc.pre_dn[i] = pd;
                if (i < n_slots) {
                    sc.e[i] = e;
                    sc.first[i] = first;
                    sc.ntot[i] = ntot;
                    // (the shared expert's slot 0 was filled at the start)
                    if (i >= d.has_shared) {
#pragma unroll
                        for (int j = 0; j < 3; ++j) { sc.p[i][j] = tab.p[e][j]; sc.fmt[i][j] = tab.fmt[e][j]; }
                    }
                }
            }
#pragma unroll
            for (int u = 0; u < 4; ++u) {
                const int i = 32 * u + lane;
                if (i < n_routed) { s_perm[i] = pv0[u]; s_wts[i] = wv0[u]; }
            }
            for (int i0 = 128; i0 < n_routed; i0 += 128) {
                int v[4];
                float wv[4];
#pragma unroll
                for (int u = 0; u < 4; ++u) {
                    const int i = i0 + 32 * u + lane;
                    v[u] = i < n_routed ? __ldcg(A.perm + i) : 0;
                    wv[u] = i < n_routed ? __ldcg(A.wts + i) : 0.0f;
                }
#pragma unroll
                for (int u = 0; u < 4; ++u) {
                    const int i = i0 + 32 * u + lane;
                    if (i < n_routed) { s_perm[i] = v[u]; s_wts[i] = wv[u]; }
                }
            }
            __syncwarp();
            n_gu = sc.pre_gu[n_slots];
            n_items = n_gu + sc.pre_dn[n_slots];
            routed = true;
            pdl_launch();
        };
        if (n_sh_items == 0) wait_routing();
        // items are handed out by one counter (zeroed per call) in the order
        // above: the shared expert's gate/up items (Q8_0, the heaviest) first,
        // so the CTAs even out on the lighter routed items that follow
        // A claim is the atomic (lane 0) and, later, the broadcast of its
        // result: nothing reads the result register before the broadcast, so
        // the atomic's round trip runs while the stages are posted.
        auto claim_issue = [&]() -> uint32_t {
            uint32_t v = 0;
            if (lane == 0) v = atomicAdd(A.next, 1u);
            return v;
        };
        auto claim_take = [&](uint32_t v) -> int { return __shfl_sync(kFull, (int)v, 0); };
        int id_next = claim_take(claim_issue());
        for (;;) {
            const int id = id_next;
            if (!routed && id >= n_sh_items) wait_routing();
            const int item = id < n_items ? id : -1;
            // claim the following item now, so that the atomic's latency hides
            // behind this item's stages; before the routing result is in, only
            // after this item's stages are posted, so that the shared expert's
            // items spread over the CTAs instead of going two to a CTA
            const bool claim_early = routed || !A.split_shared;
            const bool pending = item >= 0 && claim_early;
            const uint32_t pend = pending ? claim_issue() : 0u;
            if (item >= 0) {
                decode_item(A, sc, s_perm, n_slots, n_gu, item, cur_gu, cur_dn, P);
                fmt0 = sc.fmt[P.slot][P.down ? 2 : 0];
                fmt1 = sc.fmt[P.slot][P.down ? 2 : 1];
                const int span = P.ke - P.kb;
                const int per0 = geo[P.down][fmt0 - 1][P.ntok - 1].per, per1 = geo[0][fmt1 - 1][P.ntok - 1].per;
                P.nst0 = (span + per0 - 1) / per0;
                P.nst = P.down ? 2 * P.nst0 : P.nst0 + (span + per1 - 1) / per1;
            }
            const int nst = item >= 0 ? P.nst : 1;
            bool failed = false;
            bool h_in = !(item >= 0 && P.down);   // a down item copies h once its slot's blocks are in
            // this lane's copy for the current phase (one tensor of the item)
            const uint8_t* c_src = nullptr;
            uint32_t c_stride = 0, c_dst = 0;
            const Geo* G = nullptr;
            int fmt = 0, tensor = 0, phase_j = 0;
            for (int pj = 0; pj < nst; ++pj) {
                const int slot = p_q % kNST;
                const uint32_t full = bar0 + 8 * slot, empty = bar0 + 8 * (kNST + slot);
                if (p_q >= kNST && !mbar_wait(empty, ((p_q / kNST) & 1) ^ 1, A.err, kErrEmpty, A.wait_ns)) {
                    failed = true;
                    break;
                }
                if (!routed && p_q >= kPreRouteDepth) {
                    // Before the routing result is in, keep at most
                    // kPreRouteDepth stages in flight: the routing's own memory
                    // round trips (logits, the published result, the first
                    // routed weights) are on the step's critical path, and
                    // full queues would stretch each of them.
                    const int sq = p_q - kPreRouteDepth;
                    if (!mbar_wait(bar0 + 8 * (kNST + sq % kNST), (sq / kNST) & 1, A.err, kErrEmpty, A.wait_ns)) {
                        failed = true;
                        break;
                    }
                }
                if (A.fail_first_stage && p_q == 0) {
                    // test hook: nothing arrives on this slot's full barrier and
                    // no copy targets it, so the consumers' wait runs out
                    ++p_q;
                    if (item < 0) break;
                    continue;
                }
                if (item < 0) {   // sentinel: consumers stop here
                    if (lane == 0) { hdr[slot].item = -1; s_posted[slot] = p_q; mbar_arrive(full); }
                    ++p_q;
                    break;
                }
                if (pj == 0 || pj == P.nst0) {
                    // phases: gate then up (gate/up items); rows rb then rb + 1 (down items, tensor 2 / 3)
                    tensor = P.down ? (pj == 0 ? 2 : 3) : (pj == 0 ? 0 : 1);
                    phase_j = pj;
                    fmt = tensor == 1 ? fmt1 : fmt0;
                    G = &geo[P.down][fmt - 1][P.ntok - 1];
                    const uint8_t* tbase = sc.p[P.slot][tensor >= 2 ? 2 : tensor];
                    c_src = nullptr; c_stride = 0; c_dst = 0;
                    if (lane < G->npl) {
                        c_src = tbase + G->pl[lane] + (int64_t)(P.rb + (tensor == 3 ? 1 : 0)) * G->rbstr[lane];
                        c_stride = G->cstr[lane];
                        c_dst = G->woff[lane];
                    }
                    if (lane >= 4 && lane < 4 + 2 * P.ntok) {
                        const VecSrc& vs = P.down ? vh : vx;
                        const int tk = (lane - 4) / 2, piece = (lane - 4) - 2 * tk;
                        int v = P.vec[0];
#pragma unroll
                        for (int t2 = 1; t2 < kDecodeTok; ++t2) if (tk == t2) v = P.vec[t2];
                        const uint8_t* qv = reinterpret_cast<const uint8_t*>(vs.q + (size_t)v * vs.q_stride);
                        const uint8_t* sv = reinterpret_cast<const uint8_t*>(vs.st + (size_t)v * vs.st_stride);
                        const int fam = fmt == kQ2K || fmt == kQ3K ? kF2
                                      : fmt == kQ4K || fmt == kQ6K ? kF4 : fmt == kBF16 ? kFB : kF8;
                        const uint32_t tb = G->tok0 + tk * G->tstride;
                        if (piece == 0) { c_src = qv + (size_t)fam * vs.nsb * 512; c_stride = 512; c_dst = tb + G->tx; }
                        if (piece == 1 && fmt == kBF16) {   // the lo operands instead of statistics
                            c_src = qv + (size_t)kFBL * vs.nsb * 512; c_stride = 512; c_dst = tb + G->ts;
                        } else if (piece == 1) {
                            c_src = sv; c_stride = kStatFloats * 4; c_dst = tb + G->ts;
                        }
                    }
                }
                const int per = G->per;
                const int s0 = P.kb + (pj - phase_j) * per, ks = min(per, P.ke - s0);
                const uint32_t stage = ring + slot * slot_bytes(MT);
                const uint32_t bytes = c_src ? (uint32_t)ks * c_stride : 0u;
                uint32_t total = bytes;
#pragma unroll
                for (int off = 16; off >= 1; off >>= 1) total += __shfl_xor_sync(kFull, total, off);
                if (lane == 0) {
                    int4* H = reinterpret_cast<int4*>(&hdr[slot]);
                    H[0] = make_int4(item, pj, P.nst, s0);
                    H[1] = make_int4(ks, fmt, tensor, P.ntok);
                    H[2] = make_int4(P.rb, P.e, P.shared, P.slot);
                    H[3] = make_int4(P.asg[0], P.asg[1], P.asg[2], P.asg[3]);
                    H[4] = make_int4(P.kb, P.half, 0, 0);
                    s_posted[slot] = p_q;
                    mbar_arrive_tx(full, total);
                }
                __syncwarp();
                // weight planes (lanes 0..3) first; a down item's weights stream
                // while the last blocks of its slot's h may still be computed
                if (bytes && lane < 4) bulk_copy_hint(stage + c_dst, c_src + (size_t)s0 * c_stride, bytes, full, wpol);
                if (!h_in) {
                    // h of the slot: every gate/up item of the slot publishes its
                    // tokens' 32-row blocks (release add on the slot's counter)
                    const uint32_t target = (uint32_t)((d.I / 32) * sc.ntot[P.slot]);
                    const uint32_t* cnt = A.hready + P.slot;
                    if (lane == 0 && ld_acquire(cnt) < target) {
                        const uint64_t t0 = global_ns();
                        while (ld_acquire(cnt) < target) {
                            if (global_ns() - t0 > A.wait_ns) { atomicOr(A.err, kErrReady); s_fail = 1; break; }
                            __nanosleep(100);
                        }
                    }
                    __syncwarp();
                    // every lane that copies h acquires the counter itself, then
                    // orders its bulk (async proxy) reads after that acquire
                    if (lane >= 4) (void)ld_acquire(cnt);
                    asm volatile("fence.proxy.async.global;" ::: "memory");
                    h_in = true;
                }
                if (!tokens_in && !P.down) {
                    // the shared expert's items run before routing: wait for the
                    // prepared tokens once
                    wait_word(A.logits_done, A.n_logit_ctas);
                    tokens_in = true;
                }
                if (bytes && lane >= 4) bulk_copy(stage + c_dst, c_src + (size_t)s0 * c_stride, bytes, full);
                ++p_q;
            }
            if (failed) { if (lane == 0) { atomicOr(A.err, kErrEmpty); s_fail = 1; } break; }
            if (item < 0) break;
            id_next = claim_take(pending ? pend : claim_issue());
        }
    } else {
        // ============================ consumer warps =============================
        // warp w: row tiles rt0 .. rt0 + kNT - 1 of the stage's 32 rows and
        // superblocks col, col + kCols, ... (Q8_0: both halves of the code
        // pairs of each)
        const int rt0 = kNT == 2 ? 0 : (warp & 1), col = kNT == 2 ? warp : (warp >> 1);
        float acc[2][MT][4];   // [0] gate (or rows rb), [1] up (or rows rb + 1); rows g + 8 i
        float cur[MT][4];      // the tensor being streamed
#pragma unroll
        for (int tk = 0; tk < MT; ++tk)
#pragma unroll
            for (int i = 0; i < 4; ++i) acc[0][tk][i] = acc[1][tk][i] = cur[tk][i] = 0.0f;
        int n_done = 0;   // items finished by this CTA (selects the reduction buffer and the owner warps)
        for (int q = 0;; ++q) {
            const int slot = q % kNST;
            if (!mbar_wait(bar0 + 8 * slot, (q / kNST) & 1, A.err, kErrFull, A.wait_ns)) {
                if (lane == 0) s_fail = 1;
                break;
            }
            const Hdr& H = hdr[slot];
            if (H.item < 0) break;
            const uint32_t stage = ring + slot * slot_bytes(MT);
            const int fmt = H.fmt, ks = H.ks, ntok = H.ntok;
            const bool dn = H.tensor >= 2;
            const Geo& GS = geo[dn ? 1 : 0][fmt - 1][ntok - 1];
            // superblock jj of the stage goes to warp column (jj + s) % kCols, s the
            // stage's first superblock counted over the whole item, so every warp
            // gets the same share of an item even where a stage's count is not a
            // multiple of kCols
            const int s_item = H.s0 + ((H.tensor & 1) ? (dn ? A.nsbi : A.nsbx) : 0);
            const int wcol = (col - s_item % kCols + kCols) % kCols;
            if ((H.tensor & 1) && H.s0 == H.kb) {
                // first stage of the second phase: the first phase's sums are complete
#pragma unroll
                for (int tk = 0; tk < MT; ++tk)
#pragma unroll
                    for (int i = 0; i < 4; ++i) { acc[0][tk][i] += cur[tk][i]; cur[tk][i] = 0.0f; }
            }
            // Items of several tokens: Q2_K / Q3_K / Q4_K / Q8_0 tiles take the
            // tokens two at a time (the code operands built once for both, per
            // 16-row tile); sums equal to the per-token passes
            constexpr bool kPairs = MT > 1 && kNT == 2;
            const bool pairs = kPairs && (fmt == kQ2K || fmt == kQ3K || fmt == kQ4K || fmt == kQ80);
#pragma unroll
            for (int tk = 0; tk < MT; ++tk) {
                if (tk >= ntok) break;
                if constexpr (kPairs) {
                    if (pairs && (tk & 1)) continue;   // done with tk - 1
                    if (pairs && tk + 1 < ntok) {
                        for (int jj = wcol; jj < ks; jj += kCols) {
#pragma unroll 1
                            for (int rt = 0; rt < 2; ++rt) {
                                // this row tile's sums of the two tokens (indices fixed at compile
                                // time on this side, so the sums stay in registers)
                                float a[2][2];
#pragma unroll
                                for (int hl = 0; hl < 2; ++hl) {
                                    a[0][hl] = rt ? cur[tk][2 + hl] : cur[tk][hl];
                                    a[1][hl] = rt ? cur[(tk + 1) % MT][2 + hl] : cur[(tk + 1) % MT][hl];
                                }
                                if (fmt == kQ80) {
                                    tile_pair_q80(GS, stage, jj, 0, rt, tk, zaddr, a);
                                    tile_pair_q80(GS, stage, jj, 1, rt, tk, zaddr, a);
                                } else if (fmt == kQ2K) {
                                    tile_pair_q2k(GS, stage, jj, rt, tk, zaddr, a);
                                } else if (fmt == kQ3K) {
                                    tile_pair_q3k(GS, stage, jj, rt, tk, zaddr, a);
                                } else {
                                    tile_pair_q4k(GS, stage, jj, rt, tk, zaddr, a);
                                }
#pragma unroll
                                for (int hl = 0; hl < 2; ++hl) {
                                    if (rt) { cur[tk][2 + hl] = a[0][hl]; cur[(tk + 1) % MT][2 + hl] = a[1][hl]; }
                                    else { cur[tk][hl] = a[0][hl]; cur[(tk + 1) % MT][hl] = a[1][hl]; }
                                }
                            }
                        }
                        continue;
                    }
                }
                if (fmt == kQ80) {
                    for (int jj = wcol; jj < ks; jj += kCols) {   // both halves of each superblock's code pairs
                        TileAcc<kNT> T0, T1;
                        tile_mma<kQ80, kNT>(GS, stage, jj, 0, rt0, tk, zaddr, T0);
                        tile_epi<kQ80, kNT>(GS, stage, jj, 0, rt0, tk, T0, cur[tk]);
                        tile_mma<kQ80, kNT>(GS, stage, jj, 1, rt0, tk, zaddr, T1);
                        tile_epi<kQ80, kNT>(GS, stage, jj, 1, rt0, tk, T1, cur[tk]);
                    }
                } else if (fmt == kQ2K) {
                    tile_cols<kQ2K>(GS, stage, wcol, ks, rt0, tk, zaddr, cur[tk]);
                } else if (fmt == kQ3K) {
                    tile_cols<kQ3K>(GS, stage, wcol, ks, rt0, tk, zaddr, cur[tk]);
                } else if (fmt == kQ4K) {
                    tile_cols<kQ4K>(GS, stage, wcol, ks, rt0, tk, zaddr, cur[tk]);
                } else if (fmt == kQ6K) {
                    tile_cols<kQ6K>(GS, stage, wcol, ks, rt0, tk, zaddr, cur[tk]);
                } else {
                    tile_cols<kBF16>(GS, stage, wcol, ks, rt0, tk, zaddr, cur[tk]);
                }
            }
            // fields needed after the slot is released to the producer
            const bool item_end = H.j == H.nst - 1;
            int e_rb = 0, e_ntok = 0, e_shared = 0, e_e = 0, e_slot = 0, e_half = -1;
            int e_asg[kDecodeTok];
            if (item_end) {
                e_rb = H.rb; e_ntok = H.ntok; e_shared = H.shared; e_e = H.e; e_slot = H.slot; e_half = H.half;
#pragma unroll
                for (int tk = 0; tk < kDecodeTok; ++tk) e_asg[tk] = H.asg[tk];
            }
            __syncwarp();
            if (lane == 0) mbar_arrive(bar0 + 8 * (kNST + slot));
            if (!item_end) continue;

            // ---- item done: phase 0 (gate, or rows rb) in acc[0], phase 1 (up, or
            // rows rb + 1) still streaming in cur
            const int g = lane >> 2, t4 = lane & 3;
            const int buf = kRedBufs == 2 ? (n_done & 1) : 0;
#pragma unroll
            for (int u = 0; u < 2; ++u)
#pragma unroll
                for (int tk = 0; tk < MT; ++tk)
#pragma unroll
                    for (int i = 0; i < 2 * kNT; ++i) {
                        float v = u == 1 ? acc[u][tk][i] + cur[tk][i] : acc[u][tk][i];
                        v += __shfl_xor_sync(kFull, v, 1);
                        v += __shfl_xor_sync(kFull, v, 2);
                        if (t4 == 0) {
                            red[buf][warp][u][tk][16 * rt0 + 8 * i + g] = v;
                            if (kNT == 1) red[buf][warp][u][tk][16 * (1 - rt0) + 8 * i + g] = 0.0f;
                        }
                    }
#pragma unroll
            for (int tk = 0; tk < MT; ++tk)
#pragma unroll
                for (int i = 0; i < 4; ++i) acc[0][tk][i] = acc[1][tk][i] = cur[tk][i] = 0.0f;
            consumer_sync();
            // the finishing work of token tk goes to warp (n_done + tk) % kConsumers
            const int tk = (warp - n_done % kConsumers + kConsumers) % kConsumers;
            if (tk < e_ntok) {
                int a = e_asg[0];
#pragma unroll
                for (int t2 = 1; t2 < kDecodeTok; ++t2) if (tk == t2) a = e_asg[t2];
                // lane = row of the 32-row block
                float v0 = 0.0f, v1 = 0.0f;
#pragma unroll
                for (int c2 = 0; c2 < kConsumers; ++c2) {
                    v0 += red[buf][c2][0][tk][lane];
                    v1 += red[buf][c2][1][tk][lane];
                }
                bool finish = true;
                if (!dn && e_half >= 0) {
                    // K half of a shared-expert block: publish this half's sums; the
                    // half that counts second adds the other's (a + b, the same bits
                    // in either order) and finishes the block
                    const int t = a - d.T * d.K;   // the token (shared-expert assignment)
                    float* sp = A.spart + (size_t)t * 4 * d.I;
                    sp[(2 * e_half + 0) * d.I + 32 * e_rb + lane] = v0;
                    sp[(2 * e_half + 1) * d.I + 32 * e_rb + lane] = v1;
                    // the warp barrier orders every lane's stores before lane 0's
                    // acquire-release count, which publishes them and, in the
                    // half that counts second, acquires the other half's; the
                    // second barrier orders that acquire before every lane's loads
                    __syncwarp();
                    uint32_t before = 0;
                    if (lane == 0) before = atom_acq_rel_add(A.scount + (size_t)t * (d.I / 32) + e_rb, 1u);
                    before = __shfl_sync(kFull, before, 0);
                    __syncwarp();
                    finish = before == 1u;
                    if (finish) {
                        const int o = 1 - e_half;
                        v0 += __ldcg(sp + (2 * o + 0) * d.I + 32 * e_rb + lane);
                        v1 += __ldcg(sp + (2 * o + 1) * d.I + 32 * e_rb + lane);
                    }
                }
                if (!finish) {
                } else if (dn) {
                    A.pdn[(size_t)a * d.H + 32 * e_rb + lane] = v0;
                    A.pdn[(size_t)a * d.H + 32 * (e_rb + 1) + lane] = v1;
                } else {
                    // SwiGLU (routing weight folded in), then prepare h for the down projection
                    // routing weights: written by the logits kernel's routing CTA,
                    // acquired by this CTA's producer before it posted the item and
                    // cached in shared memory (the first kMaxCachedAssign entries)
                    const float w = e_shared ? 1.0f : a < kMaxCachedAssign ? s_wts[a] : __ldcg(A.wts + a);
                    const float hv = v0 / (1.0f + expf(-v0)) * v1 * w;
                    const int fam = families_of(sc.fmt[e_slot][2]);
                    __half* hq = A.hq + (size_t)a * kFamSlots * A.nsbi * 256;
                    float* hs = A.hs + (size_t)a * A.nsbi * kStatFloats;
                    prep_block32(hv, e_rb, fam, hq, hs, A.nsbi);
                    const int n_rb = d.I / 32;
                    if (e_rb == n_rb - 1)
                        for (int jb = n_rb; jb < 8 * A.nsbi; ++jb) prep_block32(0.0f, jb, fam, hq, hs, A.nsbi);
                    // publish the block: the warp barrier orders every lane's
                    // writes before lane 0's release add on the slot's counter
                    // (down items of the slot acquire it)
                    __syncwarp();
                    if (lane == 0) red_release_add(A.hready + e_slot, 1u);
                }
            }
            // with two buffers the next item end writes the other one and its
            // barrier orders these reads before reuse; with one, wait here
            if (kRedBufs == 1) consumer_sync();
            ++n_done;
        }
    }
    // After a wait ran out, wait (bounded) for the copies still in flight into
    // each slot before the CTA exits.  Without a failure every posted stage
    // has been consumed, so nothing is in flight.
    __syncthreads();
    if (warp == kProducerWarp && s_fail && lane < kNST && s_posted[lane] >= 0)
        mbar_wait(bar0 + 8 * lane, (s_posted[lane] / kNST) & 1, A.err, kErrFull, A.wait_ns);
}

// out[t] = sum of the token's routed expert outputs in slot order, then the
// shared expert (deterministic order; routing weights are folded into h)
__global__ void combine_kernel(Dims d, const float* __restrict__ pdn, float* __restrict__ out) {
    pdl_wait();
    pdl_launch();
    const int r = blockIdx.x * blockDim.x + threadIdx.x;
    if (r >= d.H) return;
    for (int t = blockIdx.y; t < d.T; t += gridDim.y) {
        float y = 0.0f;
        for (int j = 0; j < d.K; ++j) y += __ldg(pdn + (size_t)(t * d.K + j) * d.H + r);
        if (d.has_shared) y += __ldg(pdn + (size_t)(d.T * d.K + t) * d.H + r);
        out[(size_t)t * d.H + r] = y;
    }
}

void decode_setup() {
    cudaFuncSetAttribute(ffn_kernel<1>, cudaFuncAttributeMaxDynamicSharedMemorySize, ring_bytes(1));
    cudaFuncSetAttribute(ffn_kernel<kDecodeTok>, cudaFuncAttributeMaxDynamicSharedMemorySize, ring_bytes(kDecodeTok));
}

void combine_setup() { prefer_max_shared(combine_kernel); }

}  // namespace

size_t decode_counter_bytes(const Dims& d) {
    // the item counter, one h counter per expert slot, then one half-count per
    // (token, 32-row block) of the shared expert's K-split gate/up blocks
    return 4 + 4 * (kMaxExperts + 1) + 4 * (size_t)d.T * (d.I / 32);
}

cudaError_t launch_decode_mma(const Dims& d, const ExpertTab& tab, const Work& w, float* out, cudaStream_t s) {
    if (d.T == 0) return cudaSuccess;
    const int num_sms = device_setup(kSetupDecode, decode_setup);
    if (num_sms <= 0) return cudaErrorInvalidDevice;
    DecodeArgs A;
    A.d = d;
    A.nsbx = (d.H + 255) / 256;
    A.nsbi = (d.I + 255) / 256;
    A.xq = w.xq; A.xs = w.xs; A.hq = w.hq; A.hs = w.hs;
    A.perm = w.perm; A.wts = w.wts;
    A.plan = w.plan;
    A.pdn = w.pdn;
    A.next = w.counters;
    A.hready = w.counters + 1;
    A.scount = w.counters + 1 + (kMaxExperts + 1);
    A.spart = w.spart;
    A.split_shared = MQ_SPLIT_SHARED && d.T == 1 && d.has_shared && A.nsbx >= 2 ? 1 : 0;   // one token: the routing front
    A.logits_done = w.logits_done;
    A.route_ready = w.route_ready;
    A.n_logit_ctas = router_logits_ctas(d);   // the logits kernel's grid
    A.err = w.err;
    A.wait_ns = 1000000000ull;
    A.fail_first_stage = 0;
    uint64_t test_ns = 0;
    if (take_wait_test(&test_ns)) { A.wait_ns = test_ns; A.fail_first_stage = 1; }
    // one token: every item carries one, and the accumulators shrink to one token's
    const bool one = d.T == 1;
    const int smem = ring_bytes(one ? 1 : kDecodeTok);
    for (int dn = 0; dn < 2; ++dn)
        for (int f = 1; f <= kNumFormats; ++f)
            for (int n = 1; n <= kDecodeTok; ++n)
                make_geo(A.geo[dn][f - 1][n - 1], d, dn == 1, f, n, slot_bytes(one ? 1 : kDecodeTok));
    prof_begin("ffn_mma", s);
    cudaError_t err = one ? launch_pdl(ffn_kernel<1>, dim3(num_sms), dim3(kThreads), smem, s, tab, A)
                          : launch_pdl(ffn_kernel<kDecodeTok>, dim3(num_sms), dim3(kThreads), smem, s, tab, A);
    prof_end(s);
    if (err != cudaSuccess) return err;
    return launch_combine(d, w.pdn, out, s);
}

cudaError_t launch_combine(const Dims& d, const float* pdn, float* out, cudaStream_t s) {
    if (device_setup(kSetupCombine, combine_setup) <= 0) return cudaErrorInvalidDevice;
    prof_begin("combine", s);
    // one CTA row per token (up to 65535; the kernel strides over the rest),
    // so large batches stream the partial outputs at full bandwidth
    const cudaError_t err = launch_pdl(combine_kernel, dim3((d.H + 255) / 256, d.T < 65535 ? d.T : 65535), dim3(256),
                                       0, s, d, pdn, out);
    prof_end(s);
    return err;
}

}  // namespace mq
