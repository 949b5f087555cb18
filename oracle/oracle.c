/*
 * Oracle for the quantized MoE expert FFN — TEST INFRASTRUCTURE ONLY.
 * (Plain C, compiled with -O1 -ffp-contract=off.  The default build is
 * single-threaded; a second build with -fopenmp splits independent rows and
 * tokens over threads through the `omp` pragmas below, which change no
 * row's or token's arithmetic, so both builds give identical bits.)
 *
 * Only tests/, __graft_entry__.smoke() and the benchmark's CPU-baseline leg
 * may load this code.  It shares nothing with the CUDA library.
 *
 * What each part follows, and what pins it (tests/test_oracle_*.py):
 *
 *  - Block formats (Sec. 3.3: tensors stored in llama.cpp-style k-quant
 *    block formats Q2_K/Q3_K/Q4_K/Q6_K and Q8, the planner's upgrade
 *    targets for small and medium tensors being Q8 and Q6; a bf16 format
 *    for tensors kept unquantized; Sec. 4.1 implementation details).
 *    The paper gives no byte layout, so the layout below is this project's
 *    own "-style" definition: every format blocks along the contraction
 *    (column) axis, rows are padded to whole blocks with zero weights and
 *    to whole tiles of 32 rows with zero rows, and each field lives in its
 *    own 256-byte aligned plane.  A plane lists, for each 32-row tile and
 *    each block, the field's record of the 32 rows (records longer than 64
 *    bytes are cut in 64-byte units, unit-major; see unit_at).  Code bits
 *    are placed in "pair order" (see code_pos_*: the two codes of a pair
 *    sit 16 bits apart in one word), sub-block scale fields in "slot
 *    order" (slot_of); Q8_0 codes are stored offset by 128.  Q6_K: 16
 *    sub-blocks of 16, fp16 d, an 8-bit scale per sub-block stored offset
 *    by 128, 6-bit codes q in 0..63 for the value d * sc * (q - 32), kept
 *    as a low-nibble plane (code_pos_4bit16) and a high-two-bit plane
 *    (code_pos_2bit).  BF16: 32-weight blocks of raw bf16 values in MMA
 *    fragment order (bf16_pos).
 *      PINNED by hand-built blocks (tests/golden/hand_blocks.json), by
 *      single-bit placement tests, by grid blocks that must re-pack to
 *      themselves, and by nearest-grid-point brute force on random blocks.
 *  - Quantizer (pack): deterministic rule of this project (the paper leaves
 *    the quantizer to llama.cpp's importance-matrix search, prior art).
 *      PINNED by the nearest-code brute force and grid-block round trip.
 *  - Router (Sec. 3.2: sigmoid expert scores, topk_group over the pruned
 *    experts, num_experts_per_tok = k): canonical fp32 arithmetic so that
 *    expert indices can be bit-exact across CPU and GPU.
 *      PINNED by integer-exact logits, sigmoid vs double exp (<= 4 ulp),
 *      G=1 == plain top-k, all-groups-kept == plain top-k, exact ties,
 *      and brute-force enumeration of group choices on tiny layers.
 *  - Permutation: stable counting sort.  PINNED by integer invariants.
 *  - Expert FFN, combine and shared expert (Fig. 1: routed experts weighted
 *    by the router plus an always-on shared expert; SwiGLU FFN): fp64.
 *      PINNED by brute force against a dense numpy float64 evaluation of
 *      every expert on every token, and by one-hot inputs.
 */
#include "oracle.h"

#include <math.h>
#include <stdlib.h>
#include <string.h>

/* ------------------------------------------------------------------ */
/* fp16 / bf16 conversions (IEEE binary16, round to nearest even)       */
/* ------------------------------------------------------------------ */

static float bits_to_f32(uint32_t u) { float f; memcpy(&f, &u, 4); return f; }
static uint32_t f32_to_bits(float f) { uint32_t u; memcpy(&u, &f, 4); return u; }

static float half_to_float(uint16_t h) {
    uint32_t sign = (uint32_t)(h & 0x8000u) << 16;
    uint32_t expo = (h >> 10) & 0x1fu;
    uint32_t mant = h & 0x3ffu;
    if (expo == 0) {
        /* zero or subnormal: mant * 2^-24, exact in fp32 */
        float v = (float)mant * 5.9604644775390625e-08f;
        return sign ? -v : v;
    }
    if (expo == 31) return bits_to_f32(sign | 0x7f800000u | (mant << 13));
    return bits_to_f32(sign | ((expo + 112u) << 23) | (mant << 13));
}

static uint16_t float_to_half(float f) {
    uint32_t x = f32_to_bits(f);
    uint16_t sign = (uint16_t)((x >> 16) & 0x8000u);
    uint32_t ax = x & 0x7fffffffu;
    if (ax >= 0x7f800000u) return (uint16_t)(sign | 0x7c00u | (ax > 0x7f800000u ? 0x200u : 0));
    if (ax >= 0x477ff000u) return (uint16_t)(sign | 0x7c00u); /* >= 65520 -> inf */
    if (ax <= 0x33000000u) return sign;                        /* <= 2^-25 -> 0  */
    int e = (int)(ax >> 23) - 127;
    uint32_t mant = (ax & 0x7fffffu) | 0x800000u; /* 24 significant bits */
    if (e < -14) {
        int shift = -e - 1; /* value = mant * 2^(e-23); unit 2^-24 */
        uint32_t q = mant >> shift;
        uint32_t rem = mant & ((1u << shift) - 1u);
        uint32_t halfway = 1u << (shift - 1);
        if (rem > halfway || (rem == halfway && (q & 1u))) q++;
        return (uint16_t)(sign | q);
    }
    uint32_t q = mant >> 13;
    uint32_t rem = mant & 0x1fffu;
    uint32_t h = ((uint32_t)(e + 15) << 10) | (q & 0x3ffu);
    if (rem > 0x1000u || (rem == 0x1000u && (q & 1u))) h++;
    return (uint16_t)(sign | h);
}

static float bf16_to_float(uint16_t b) { return bits_to_f32((uint32_t)b << 16); }

/* fp32 -> bf16, round to nearest even (finite inputs) */
static uint16_t float_to_bf16(float f) {
    uint32_t u = f32_to_bits(f);
    uint32_t lsb = (u >> 16) & 1u;
    return (uint16_t)((u + 0x7FFFu + lsb) >> 16);
}

/* ------------------------------------------------------------------ */
/* Format geometry                                                      */
/* ------------------------------------------------------------------ */

#define MAX_PLANES 4
#define PLANE_ALIGN 256

typedef struct {
    int qk;                 /* weights per block along the contraction axis */
    int nplanes;
    int bytes[MAX_PLANES];  /* bytes per (row, block) record in each plane */
    int unit[MAX_PLANES];   /* records are stored in units of this many bytes */
} geom;

static int get_geom(int fmt, geom* g) {
    memset(g, 0, sizeof(*g));
    switch (fmt) {
    case ORC_Q4_K: g->qk = 256; g->nplanes = 4;
        g->bytes[0] = 2; g->bytes[1] = 2; g->bytes[2] = 12; g->bytes[3] = 128;
        g->unit[0] = 2; g->unit[1] = 2; g->unit[2] = 12; g->unit[3] = 64; return 0;
    case ORC_Q2_K: g->qk = 256; g->nplanes = 4;
        g->bytes[0] = 2; g->bytes[1] = 2; g->bytes[2] = 16; g->bytes[3] = 64;
        g->unit[0] = 2; g->unit[1] = 2; g->unit[2] = 16; g->unit[3] = 64; return 0;
    case ORC_Q3_K: g->qk = 256; g->nplanes = 4;
        g->bytes[0] = 2; g->bytes[1] = 12; g->bytes[2] = 64; g->bytes[3] = 32;
        g->unit[0] = 2; g->unit[1] = 12; g->unit[2] = 64; g->unit[3] = 32; return 0;
    case ORC_Q8_0: g->qk = 32; g->nplanes = 2;
        g->bytes[0] = 2; g->bytes[1] = 32;
        g->unit[0] = 2; g->unit[1] = 32; return 0;
    case ORC_Q6_K: g->qk = 256; g->nplanes = 4;
        g->bytes[0] = 2; g->bytes[1] = 16; g->bytes[2] = 128; g->bytes[3] = 64;
        g->unit[0] = 2; g->unit[1] = 16; g->unit[2] = 64; g->unit[3] = 64; return 0;
    case ORC_BF16: g->qk = 32; g->nplanes = 1;
        g->bytes[0] = 64; g->unit[0] = 64; return 0;
    default: return -1;
    }
}

#define ROW_TILE 32

static int64_t round_up(int64_t v, int64_t a) { return (v + a - 1) / a * a; }

/* plane base offsets for a tensor with nblk (row, block) records in total,
   rows counted after padding to whole 32-row tiles */
static void plane_offsets(const geom* g, int64_t nblk, int64_t off[MAX_PLANES + 1]) {
    off[0] = 0;
    for (int p = 0; p < g->nplanes; p++)
        off[p + 1] = off[p] + round_up(nblk * g->bytes[p], PLANE_ALIGN);
}

/* Byte offset, inside plane p, of unit u of the record (row r, block b):
   records are grouped in tiles of 32 rows; a plane lists, for each tile,
   each block, each unit of the record, the 32 rows of the tile. */
static int64_t unit_at(const geom* g, int p, int64_t nb, int64_t r, int64_t b, int u) {
    int64_t nu = g->bytes[p] / g->unit[p];
    return ((((r / ROW_TILE) * nb + b) * nu + u) * ROW_TILE + r % ROW_TILE) * g->unit[p];
}

size_t oracle_packed_size(int fmt, int64_t rows, int64_t cols) {
    geom g;
    if (get_geom(fmt, &g) || rows < 0 || cols < 0) return 0;
    int64_t nb = (cols + g.qk - 1) / g.qk;
    int64_t off[MAX_PLANES + 1];
    plane_offsets(&g, round_up(rows, ROW_TILE) * nb, off);
    return (size_t)off[g.nplanes];
}

/* ------------------------------------------------------------------ */
/* Positions of fields inside a block                                   */
/* ------------------------------------------------------------------ */
/* Codes are stored in little-endian 32-bit words; these functions give
 * (word index, bit position) of the code of weight k of a block.  A block
 * is cut in sub-blocks of n weights (n = 16 for the 2-bit / 1-bit codes of
 * Q2_K and Q3_K, 32 for Q4_K and for a Q8_0 block):
 *   j = k / n  (sub-block),  p = k % n,  m = p / 2,  e = p % 2,
 * so each sub-block is a sequence of code pairs m = 0, 1, ... and the two
 * codes of a pair (e = 0, 1) always sit 16 bits apart in one word. */

/* 2-bit codes (Q2_K codes, low two bits of Q3_K codes): 16 words/block.
   Word 4 (j % 4) + j / 4 holds sub-block j; pair m at bit 2 m (+16 e). */
static void code_pos_2bit(int k, int* word, int* bit) {
    int j = k >> 4, p = k & 15, m = p >> 1, e = p & 1;
    *word = 4 * (j & 3) + (j >> 2);
    *bit = 16 * e + 2 * m;
}

/* 1-bit plane (high bit of Q3_K codes): 8 words/block.  Word
   2 (j % 4) + j / 8 holds sub-blocks j with equal j % 4 and j / 8; the one
   with (j / 4) % 2 = 1 takes the upper byte of each 16-bit half. */
static void code_pos_1bit(int k, int* word, int* bit) {
    int j = k >> 4, p = k & 15, m = p >> 1, e = p & 1;
    *word = 2 * (j & 3) + (j >> 3);
    *bit = 16 * e + 8 * ((j >> 2) & 1) + m;
}

/* 4-bit codes (Q4_K, 8 sub-blocks of 32): 32 words/block, stored as two
   64-byte units (unit = j / 4).  Sub-block j takes words
   16 (j / 4) + 4 (j % 4) + 0..3; pair m at word m / 4, bit 4 (m % 4). */
static void code_pos_4bit(int k, int* word, int* bit) {
    int j = k >> 5, p = k & 31, m = p >> 1, e = p & 1;
    *word = 16 * (j >> 2) + 4 * (j & 3) + (m >> 2);
    *bit = 16 * e + 4 * (m & 3);
}

/* 8-bit codes (Q8_0, 32-weight block): 8 words/block; pair m at word m / 2,
   bit 8 (m % 2).  The stored byte is q + 128 (offset binary). */
static void code_pos_8bit(int k, int* word, int* bit) {
    int m = k >> 1, e = k & 1;
    *word = m >> 1;
    *bit = 16 * e + 8 * (m & 1);
}

/* 4-bit codes of 16-wide sub-blocks (Q6_K low nibbles): 32 words/block,
   two 64-byte units (unit = j / 8).  Sub-block j takes words
   16 (j / 8) + 4 (j % 4) + 2 ((j / 4) % 2) + 0..1; pair m at word m / 4,
   bit 4 (m % 4). */
static void code_pos_4bit16(int k, int* word, int* bit) {
    int j = k >> 4, p = k & 15, m = p >> 1, e = p & 1;
    *word = 16 * (j >> 3) + 4 * (j & 3) + 2 * ((j >> 2) & 1) + (m >> 2);
    *bit = 16 * e + 4 * (m & 3);
}

/* BF16 block of 32: position (in 16-bit units) of weight k, so that the
   four words a tensor-core fragment takes for k = 2t, 2t+1, 8+2t, 9+2t,
   16+2t, 17+2t, 24+2t, 25+2t are contiguous. */
static int bf16_pos(int k) { return 8 * ((k & 7) >> 1) + 2 * (k >> 3) + (k & 1); }

static uint32_t get_word(const uint8_t* p, int w) {
    const uint8_t* b = p + 4 * w;
    return (uint32_t)b[0] | ((uint32_t)b[1] << 8) | ((uint32_t)b[2] << 16) | ((uint32_t)b[3] << 24);
}

static uint32_t get_field(const uint8_t* p, int word, int bit, int width) {
    return (get_word(p, word) >> bit) & ((1u << width) - 1u);
}

static void put_field(uint8_t* p, int word, int bit, int width, uint32_t v) {
    uint32_t w = get_word(p, word);
    uint32_t mask = ((1u << width) - 1u) << bit;
    w = (w & ~mask) | ((v << bit) & mask);
    uint8_t* b = p + 4 * word;
    b[0] = (uint8_t)w; b[1] = (uint8_t)(w >> 8); b[2] = (uint8_t)(w >> 16); b[3] = (uint8_t)(w >> 24);
}

/* Slot order of the 16 sub-blocks of Q2_K / Q3_K. */
static int slot_of(int j) {
    int n = j & 7, tile = j >> 3;
    return 4 * (n >> 1) + 2 * tile + (n & 1);
}

static uint16_t rd16(const uint8_t* p) { return (uint16_t)(p[0] | (p[1] << 8)); }
static void wr16(uint8_t* p, uint16_t v) { p[0] = (uint8_t)v; p[1] = (uint8_t)(v >> 8); }

/* Q3_K scale field of sub-block j (6 bits, stored value = sc + 32) */
static int q3_get_scale(const uint8_t* s, int j) {
    int u = slot_of(j);
    int lo = (s[u >> 1] >> (4 * (u & 1))) & 15;
    int hi = (s[8 + (u >> 2)] >> (2 * (u & 3))) & 3;
    return lo | (hi << 4);
}
static void q3_put_scale(uint8_t* s, int j, int v) {
    int u = slot_of(j);
    s[u >> 1] = (uint8_t)((s[u >> 1] & ~(15 << (4 * (u & 1)))) | ((v & 15) << (4 * (u & 1))));
    s[8 + (u >> 2)] = (uint8_t)((s[8 + (u >> 2)] & ~(3 << (2 * (u & 3)))) | (((v >> 4) & 3) << (2 * (u & 3))));
}

/* Q4_K scale/min fields of sub-block j (6 bits each) */
static void q4_get(const uint8_t* s, int j, int* sc, int* m) {
    uint32_t hi = (uint32_t)s[8] | ((uint32_t)s[9] << 8) | ((uint32_t)s[10] << 16) | ((uint32_t)s[11] << 24);
    *sc = (s[j] & 15) | (int)(((hi >> (4 * j)) & 3) << 4);
    *m = (s[j] >> 4) | (int)(((hi >> (4 * j + 2)) & 3) << 4);
}
static void q4_put(uint8_t* s, int j, int sc, int m) {
    s[j] = (uint8_t)((sc & 15) | ((m & 15) << 4));
    uint32_t hi = (uint32_t)s[8] | ((uint32_t)s[9] << 8) | ((uint32_t)s[10] << 16) | ((uint32_t)s[11] << 24);
    hi &= ~(15u << (4 * j));
    hi |= ((uint32_t)((sc >> 4) & 3) << (4 * j)) | ((uint32_t)((m >> 4) & 3) << (4 * j + 2));
    s[8] = (uint8_t)hi; s[9] = (uint8_t)(hi >> 8); s[10] = (uint8_t)(hi >> 16); s[11] = (uint8_t)(hi >> 24);
}

/* ------------------------------------------------------------------ */
/* Quantizer                                                            */
/* ------------------------------------------------------------------ */

static int clampi(int v, int lo, int hi) { return v < lo ? lo : (v > hi ? hi : v); }
static int rn(float v) { return (int)nearbyintf(v); }   /* ties to even */

/* asymmetric k-quant: sub-blocks of `sublen`, codes 0..L, 6/4-bit fields 0..S */
static void quant_asym(const float* wb, int nsub, int sublen, int L, int S,
                       uint16_t* dh, uint16_t* mh, int* sc, int* m, int* q) {
    float scale[16], mn[16], max_scale = 0.0f, max_mn = 0.0f;
    for (int j = 0; j < nsub; j++) {
        float lo = 0.0f, hi = wb[j * sublen];
        for (int i = 0; i < sublen; i++) {
            float v = wb[j * sublen + i];
            if (v < lo) lo = v;
            if (v > hi) hi = v;
        }
        scale[j] = (hi - lo) / (float)L;
        mn[j] = 0.0f - lo;
        if (scale[j] > max_scale) max_scale = scale[j];
        if (mn[j] > max_mn) max_mn = mn[j];
    }
    *dh = float_to_half(max_scale / (float)S);
    *mh = float_to_half(max_mn / (float)S);
    float df = half_to_float(*dh), mf = half_to_float(*mh);
    for (int j = 0; j < nsub; j++) {
        sc[j] = df > 0.0f ? clampi(rn(scale[j] / df), 0, S) : 0;
        m[j] = mf > 0.0f ? clampi(rn(mn[j] / mf), 0, S) : 0;
        float den = df * (float)sc[j];
        float off = mf * (float)m[j];
        for (int i = 0; i < sublen; i++) {
            float num = wb[j * sublen + i] + off;
            q[j * sublen + i] = den > 0.0f ? clampi(rn(num / den), 0, L) : 0;
        }
    }
}

int oracle_pack(int fmt, const float* w, int64_t rows, int64_t cols,
                uint8_t* dst, size_t dst_bytes) {
    geom g;
    if (get_geom(fmt, &g) || !dst || (rows * cols > 0 && !w) || rows < 0 || cols < 0) return -1;
    size_t need = oracle_packed_size(fmt, rows, cols);
    if (dst_bytes < need) return -1;
    for (int64_t i = 0; i < rows * cols; i++)
        if (!isfinite(w[i])) return -2;
    memset(dst, 0, need);
    int64_t nb = (cols + g.qk - 1) / g.qk, prow = round_up(rows, ROW_TILE);
    int64_t off[MAX_PLANES + 1];
    plane_offsets(&g, prow * nb, off);
    float wb[256];
    int q[256], sc[16], m[16];
    uint8_t rec[MAX_PLANES][128];
    /* padding rows (up to a whole tile) are quantized zero rows */
    for (int64_t r = 0; r < prow; r++) {
        for (int64_t b = 0; b < nb; b++) {
            for (int k = 0; k < g.qk; k++) {
                int64_t c = b * g.qk + k;
                wb[k] = (r < rows && c < cols) ? w[r * cols + c] : 0.0f;
            }
            memset(rec, 0, sizeof(rec));
            if (fmt == ORC_Q4_K || fmt == ORC_Q2_K) {
                int is4 = fmt == ORC_Q4_K;
                uint16_t dh, mh;
                quant_asym(wb, is4 ? 8 : 16, is4 ? 32 : 16, is4 ? 15 : 3, is4 ? 63 : 15,
                           &dh, &mh, sc, m, q);
                wr16(rec[0], dh);
                wr16(rec[1], mh);
                if (is4) {
                    for (int j = 0; j < 8; j++) q4_put(rec[2], j, sc[j], m[j]);
                    for (int k = 0; k < 256; k++) { int wd, bt; code_pos_4bit(k, &wd, &bt); put_field(rec[3], wd, bt, 4, (uint32_t)q[k]); }
                } else {
                    for (int j = 0; j < 16; j++) rec[2][slot_of(j)] = (uint8_t)(sc[j] | (m[j] << 4));
                    for (int k = 0; k < 256; k++) { int wd, bt; code_pos_2bit(k, &wd, &bt); put_field(rec[3], wd, bt, 2, (uint32_t)q[k]); }
                }
            } else if (fmt == ORC_Q3_K) {
                float scale[16], maxabs = 0.0f;
                for (int j = 0; j < 16; j++) {
                    float amax = wb[16 * j];
                    for (int i = 1; i < 16; i++)
                        if (fabsf(wb[16 * j + i]) > fabsf(amax)) amax = wb[16 * j + i];
                    scale[j] = amax / -4.0f;
                    if (fabsf(scale[j]) > maxabs) maxabs = fabsf(scale[j]);
                }
                uint16_t dh = float_to_half(maxabs / 31.0f);
                float df = half_to_float(dh);
                wr16(rec[0], dh);
                for (int j = 0; j < 16; j++) {
                    int scj = df > 0.0f ? clampi(rn(scale[j] / df), -32, 31) : 0;
                    q3_put_scale(rec[1], j, scj + 32);
                    float den = df * (float)scj;
                    for (int i = 0; i < 16; i++) {
                        int k = 16 * j + i;
                        int qi = den != 0.0f ? clampi(rn(wb[k] / den), -4, 3) : 0;
                        int code = qi + 4;
                        int wd, bt;
                        code_pos_2bit(k, &wd, &bt); put_field(rec[2], wd, bt, 2, (uint32_t)(code & 3));
                        code_pos_1bit(k, &wd, &bt); put_field(rec[3], wd, bt, 1, (uint32_t)(code >> 2));
                    }
                }
            } else if (fmt == ORC_Q6_K) {
                /* symmetric: per sub-block the element of largest |w| maps to
                   code -32; 8-bit sub-block scales against d = max|scale| / 127 */
                float scale[16], maxabs = 0.0f;
                for (int j = 0; j < 16; j++) {
                    float amax = wb[16 * j];
                    for (int i = 1; i < 16; i++)
                        if (fabsf(wb[16 * j + i]) > fabsf(amax)) amax = wb[16 * j + i];
                    scale[j] = amax / -32.0f;
                    if (fabsf(scale[j]) > maxabs) maxabs = fabsf(scale[j]);
                }
                uint16_t dh = float_to_half(maxabs / 127.0f);
                float df = half_to_float(dh);
                wr16(rec[0], dh);
                for (int j = 0; j < 16; j++) {
                    int scj = df > 0.0f ? clampi(rn(scale[j] / df), -128, 127) : 0;
                    rec[1][slot_of(j)] = (uint8_t)(scj + 128);
                    float den = df * (float)scj;
                    for (int i = 0; i < 16; i++) {
                        int k = 16 * j + i;
                        int qi = den != 0.0f ? clampi(rn(wb[k] / den), -32, 31) : 0;
                        int code = qi + 32;
                        int wd, bt;
                        code_pos_4bit16(k, &wd, &bt); put_field(rec[2], wd, bt, 4, (uint32_t)(code & 15));
                        code_pos_2bit(k, &wd, &bt); put_field(rec[3], wd, bt, 2, (uint32_t)(code >> 4));
                    }
                }
            } else if (fmt == ORC_BF16) {
                for (int k = 0; k < 32; k++) {
                    uint16_t h = float_to_bf16(wb[k]);
                    if ((h & 0x7F80u) == 0x7F80u) return -2;   /* rounds beyond the bf16 range */
                    wr16(rec[0] + 2 * bf16_pos(k), h);
                }
            } else { /* Q8_0 */
                float amax = 0.0f;
                for (int k = 0; k < 32; k++) if (fabsf(wb[k]) > amax) amax = fabsf(wb[k]);
                uint16_t dh = float_to_half(amax / 127.0f);
                float df = half_to_float(dh);
                wr16(rec[0], dh);
                for (int k = 0; k < 32; k++) {
                    int qi = df > 0.0f ? clampi(rn(wb[k] / df), -127, 127) : 0;
                    int wd, bt; code_pos_8bit(k, &wd, &bt);
                    put_field(rec[1], wd, bt, 8, (uint32_t)(qi + 128));
                }
            }
            for (int p = 0; p < g.nplanes; p++)
                for (int u = 0; u < g.bytes[p] / g.unit[p]; u++)
                    memcpy(dst + off[p] + unit_at(&g, p, nb, r, b, u), rec[p] + u * g.unit[p], (size_t)g.unit[p]);
        }
    }
    return 0;
}

/* ------------------------------------------------------------------ */
/* Dequantizer                                                          */
/* ------------------------------------------------------------------ */

int oracle_unpack(int fmt, const uint8_t* src, int64_t rows, int64_t cols, float* dst) {
    geom g;
    if (get_geom(fmt, &g) || !src || !dst || rows < 0 || cols < 0) return -1;
    int64_t nb = (cols + g.qk - 1) / g.qk, prow = round_up(rows, ROW_TILE);
    int64_t off[MAX_PLANES + 1];
    plane_offsets(&g, prow * nb, off);
    /* rows are independent: the OpenMP build splits them over threads */
#pragma omp parallel for schedule(static)
    for (int64_t r = 0; r < rows; r++) {
        uint8_t rec[MAX_PLANES][128];
        for (int64_t b = 0; b < nb; b++) {
            /* gather the record of (row r, block b) from its units */
            for (int p = 0; p < g.nplanes; p++)
                for (int u = 0; u < g.bytes[p] / g.unit[p]; u++)
                    memcpy(rec[p] + u * g.unit[p], src + off[p] + unit_at(&g, p, nb, r, b, u), (size_t)g.unit[p]);
            for (int k = 0; k < g.qk; k++) {
                int64_t c = b * g.qk + k;
                if (c >= cols) break;
                float v;
                int wd, bt;
                if (fmt == ORC_Q4_K) {
                    float df = half_to_float(rd16(rec[0]));
                    float mf = half_to_float(rd16(rec[1]));
                    int sc, m; q4_get(rec[2], k / 32, &sc, &m);
                    code_pos_4bit(k, &wd, &bt);
                    int q = (int)get_field(rec[3], wd, bt, 4);
                    v = (df * (float)sc) * (float)q - mf * (float)m;
                } else if (fmt == ORC_Q2_K) {
                    float df = half_to_float(rd16(rec[0]));
                    float mf = half_to_float(rd16(rec[1]));
                    uint8_t s = rec[2][slot_of(k / 16)];
                    int sc = s & 15, m = s >> 4;
                    code_pos_2bit(k, &wd, &bt);
                    int q = (int)get_field(rec[3], wd, bt, 2);
                    v = (df * (float)sc) * (float)q - mf * (float)m;
                } else if (fmt == ORC_Q3_K) {
                    float df = half_to_float(rd16(rec[0]));
                    int s = q3_get_scale(rec[1], k / 16);
                    code_pos_2bit(k, &wd, &bt);
                    int lo = (int)get_field(rec[2], wd, bt, 2);
                    code_pos_1bit(k, &wd, &bt);
                    int hi = (int)get_field(rec[3], wd, bt, 1);
                    int q = lo | (hi << 2);
                    v = (df * (float)(s - 32)) * (float)(q - 4);
                } else if (fmt == ORC_Q6_K) {
                    float df = half_to_float(rd16(rec[0]));
                    int s = (int)rec[1][slot_of(k / 16)] - 128;
                    code_pos_4bit16(k, &wd, &bt);
                    int lo = (int)get_field(rec[2], wd, bt, 4);
                    code_pos_2bit(k, &wd, &bt);
                    int hi = (int)get_field(rec[3], wd, bt, 2);
                    int q = lo | (hi << 4);
                    v = (df * (float)s) * (float)(q - 32);
                } else if (fmt == ORC_BF16) {
                    v = bf16_to_float(rd16(rec[0] + 2 * bf16_pos(k)));
                } else {
                    float df = half_to_float(rd16(rec[0]));
                    code_pos_8bit(k, &wd, &bt);
                    int q = (int)get_field(rec[1], wd, bt, 8) - 128;
                    v = df * (float)q;
                }
                dst[r * cols + c] = v;
            }
        }
    }
    return 0;
}

/* ------------------------------------------------------------------ */
/* Router                                                               */
/* ------------------------------------------------------------------ */
/* Canonical sigmoid: s = 1 / (1 + e^-z).  e^a is computed by Cody-Waite
 * range reduction a = n ln2 + r (n = rint(a log2 e), ln2 split in a high
 * part with trailing zeros and a low part), a degree-7 Taylor polynomial
 * for e^r in Horner form with coefficients 1/i! rounded to fp32, and an
 * exact scaling by 2^n.  a is clamped to [-87, 87] so 2^n stays normal. */
static const float LOG2E_F = 0x1.715476p+0f;
static const float LN2_HI_F = 0x1.62e4p-1f;
static const float LN2_LO_F = 0x1.7f7d1cp-20f;
static const float TAYLOR[8] = {
    0x1.0p+0f, 0x1.0p+0f, 0x1.0p-1f, 0x1.555556p-3f,
    0x1.555556p-5f, 0x1.111112p-7f, 0x1.6c16c2p-10f, 0x1.a01a02p-13f,
};

float oracle_sigmoid(float z) {
    float a = 0.0f - z;
    if (a > 87.0f) a = 87.0f;
    if (a < -87.0f) a = -87.0f;
    float n = nearbyintf(a * LOG2E_F);
    float r = fmaf(-n, LN2_HI_F, a);
    r = fmaf(-n, LN2_LO_F, r);
    float p = TAYLOR[7];
    for (int i = 6; i >= 0; i--) p = fmaf(p, r, TAYLOR[i]);
    float scale = bits_to_f32((uint32_t)((int)n + 127) << 23);
    float e = p * scale;
    return 1.0f / (1.0f + e);
}

/* Canonical logit.  hidden is a multiple of 128.  The row is cut in
 * segments of 8 chunks of 128 elements.  In a segment, 32 "lanes" each
 * run one fmaf chain: chunk i ascending, then c = 0..3 over element
 * 128 i + 4 lane + c.  The 32 partials are combined by an xor butterfly
 * (offsets 16, 8, 4, 2, 1; every lane adds its partner), after which all
 * lanes hold the same value r_seg.  The logit is r_0 + r_1 + ... summed
 * left to right. */
float oracle_router_logit(const uint16_t* x, const float* w, int32_t hidden) {
    int nchunk = hidden / 128;
    float z = 0.0f;
    for (int seg = 0; seg * 8 < nchunk; seg++) {
        float acc[32], nxt[32];
        for (int l = 0; l < 32; l++) acc[l] = 0.0f;
        int iend = seg * 8 + 8 < nchunk ? seg * 8 + 8 : nchunk;
        for (int i = seg * 8; i < iend; i++)
            for (int l = 0; l < 32; l++)
                for (int c = 0; c < 4; c++) {
                    int k = i * 128 + 4 * l + c;
                    acc[l] = fmaf(bf16_to_float(x[k]), w[k], acc[l]);
                }
        for (int off = 16; off >= 1; off >>= 1) {
            for (int l = 0; l < 32; l++) nxt[l] = acc[l] + acc[l ^ off];
            for (int l = 0; l < 32; l++) acc[l] = nxt[l];
        }
        z = seg == 0 ? acc[0] : z + acc[0];
    }
    return z;
}

static int check_layer(const oracle_layer* L) {
    if (!L) return -1;
    if (L->hidden <= 0 || L->hidden % 128 || L->inter <= 0) return -1;
    if (L->n_experts <= 0 || L->n_groups <= 0 || L->n_experts % L->n_groups) return -1;
    if (L->topk_group <= 0 || L->topk_group > L->n_groups) return -1;
    if (L->top_k <= 0 || L->top_k > (L->n_experts / L->n_groups) * L->topk_group) return -1;
    return 0;
}

/* Route one token given its scores s[E] and biased scores u[E]. */
static void select_token(const oracle_layer* L, const float* s, const float* u,
                         int32_t* idx, float* w) {
    int E = L->n_experts, G = L->n_groups, gs = E / G;
    float gscore[256];
    int gkept[256];
    for (int g = 0; g < G; g++) {
        /* group score: the two largest u in the group added (one if gs == 1) */
        float top1 = -INFINITY, top2 = -INFINITY;
        for (int i = 0; i < gs; i++) {
            float v = u[g * gs + i];
            if (v > top1) { top2 = top1; top1 = v; }
            else if (v > top2) top2 = v;
        }
        gscore[g] = gs == 1 ? top1 : top1 + top2;
        gkept[g] = 0;
    }
    /* keep topk_group groups: repeated argmax, ties to the lower index */
    for (int r = 0; r < L->topk_group; r++) {
        int best = -1;
        for (int g = 0; g < G; g++)
            if (!gkept[g] && (best < 0 || gscore[g] > gscore[best])) best = g;
        gkept[best] = 1;
    }
    /* top_k experts among kept groups by u: repeated argmax, ties lower */
    int taken[1024];
    for (int e = 0; e < E; e++) taken[e] = 0;
    for (int j = 0; j < L->top_k; j++) {
        int best = -1;
        for (int e = 0; e < E; e++)
            if (gkept[e / gs] && !taken[e] && (best < 0 || u[e] > u[best])) best = e;
        taken[best] = 1;
        idx[j] = best;
    }
    /* normalised weights from the unbiased scores, summed in slot order */
    float sum = 0.0f;
    for (int j = 0; j < L->top_k; j++) sum = sum + s[idx[j]];
    for (int j = 0; j < L->top_k; j++) w[j] = (s[idx[j]] / sum) * L->routed_scale;
}

int oracle_route(const oracle_layer* L, int32_t T, const uint16_t* x,
                 const float* router_w, const float* bias, int32_t* idx,
                 float* w, float* z_out, float* s_out) {
    if (check_layer(L) || T < 0 || L->n_experts > 1024 || L->n_groups > 256) return -1;
    int E = L->n_experts, H = L->hidden;
    /* tokens are independent: the OpenMP build splits them over threads */
#pragma omp parallel
    {
    float* s = (float*)malloc(sizeof(float) * E);
    float* u = (float*)malloc(sizeof(float) * E);
#pragma omp for schedule(static)
    for (int t = 0; t < T; t++) {
        for (int e = 0; e < E; e++) {
            float z = oracle_router_logit(x + (int64_t)t * H, router_w + (int64_t)e * H, H);
            s[e] = oracle_sigmoid(z);
            u[e] = s[e] + (bias ? bias[e] : 0.0f);
            if (z_out) z_out[(int64_t)t * E + e] = z;
            if (s_out) s_out[(int64_t)t * E + e] = s[e];
        }
        select_token(L, s, u, idx + (int64_t)t * L->top_k, w + (int64_t)t * L->top_k);
    }
    free(s); free(u);
    }
    return 0;
}

int oracle_select(const oracle_layer* L, int32_t T, const float* s, const float* bias,
                  int32_t* idx, float* w) {
    if (check_layer(L) || T < 0 || L->n_experts > 1024 || L->n_groups > 256 || !s) return -1;
    int E = L->n_experts;
#pragma omp parallel
    {
    float* u = (float*)malloc(sizeof(float) * E);
#pragma omp for schedule(static)
    for (int t = 0; t < T; t++) {
        const float* st = s + (int64_t)t * E;
        for (int e = 0; e < E; e++) u[e] = st[e] + (bias ? bias[e] : 0.0f);
        select_token(L, st, u, idx + (int64_t)t * L->top_k, w + (int64_t)t * L->top_k);
    }
    free(u);
    }
    return 0;
}

int oracle_permute(int32_t T, int32_t k, int32_t E, const int32_t* idx,
                   int32_t* offsets, int32_t* perm, int32_t* inv) {
    int64_t n = (int64_t)T * k;
    for (int e = 0; e <= E; e++) offsets[e] = 0;
    for (int64_t a = 0; a < n; a++) {
        if (idx[a] < 0 || idx[a] >= E) return -1;
        offsets[idx[a] + 1]++;
    }
    for (int e = 0; e < E; e++) offsets[e + 1] += offsets[e];
    int32_t* cursor = (int32_t*)malloc(sizeof(int32_t) * (E + 1));
    for (int e = 0; e < E; e++) cursor[e] = offsets[e];
    for (int64_t a = 0; a < n; a++) {
        int32_t pos = cursor[idx[a]]++;
        perm[pos] = (int32_t)a;
        inv[a] = pos;
    }
    free(cursor);
    return 0;
}

/* ------------------------------------------------------------------ */
/* Expert FFN (fp64)                                                    */
/* ------------------------------------------------------------------ */

static double silu(double v) { return v / (1.0 + exp(-v)); }

/* y[H] += wt * down( silu(gate x) * (up x) ) for one token, all fp64 */
static void expert_apply(int H, int I, const float* Wg, const float* Wu,
                         const float* Wd, const double* x, double wt,
                         double* hbuf, double* y) {
    /* every output row is one dot product in a fixed order; the OpenMP build
     * splits the rows over threads without changing any row's arithmetic */
#pragma omp parallel for schedule(static)
    for (int i = 0; i < I; i++) {
        double g = 0.0, u = 0.0;
        const float* rg = Wg + (int64_t)i * H;
        const float* ru = Wu + (int64_t)i * H;
        for (int c = 0; c < H; c++) { g += (double)rg[c] * x[c]; u += (double)ru[c] * x[c]; }
        hbuf[i] = silu(g) * u;
    }
#pragma omp parallel for schedule(static)
    for (int r = 0; r < H; r++) {
        double o = 0.0;
        const float* rd = Wd + (int64_t)r * I;
        for (int i = 0; i < I; i++) o += (double)rd[i] * hbuf[i];
        y[r] += wt * o;
    }
}

int oracle_moe_forward(const oracle_layer* L, int32_t T, const uint16_t* x,
                       const float* router_w, const float* bias,
                       const void* const* gate, const void* const* up,
                       const void* const* down, const uint8_t* fmt,
                       float* y, int32_t* idx, float* w) {
    if (check_layer(L) || T < 0 || !y) return -1;
    int E = L->n_experts, H = L->hidden, I = L->inter, K = L->top_k;
    int nexp = E + (L->has_shared ? 1 : 0);
    int32_t* ridx = (int32_t*)malloc(sizeof(int32_t) * ((size_t)T * K + 1));
    float* rw = (float*)malloc(sizeof(float) * ((size_t)T * K + 1));
    if (oracle_route(L, T, x, router_w, bias, ridx, rw, NULL, NULL)) { free(ridx); free(rw); return -1; }
    double* xd = (double*)malloc(sizeof(double) * (size_t)T * H);
    double* yd = (double*)calloc((size_t)T * H, sizeof(double));
    double* hbuf = (double*)malloc(sizeof(double) * I);
    float* Wg = (float*)malloc(sizeof(float) * (size_t)I * H);
    float* Wu = (float*)malloc(sizeof(float) * (size_t)I * H);
    float* Wd = (float*)malloc(sizeof(float) * (size_t)H * I);
    for (int64_t i = 0; i < (int64_t)T * H; i++) xd[i] = (double)bf16_to_float(x[i]);
    int rc = 0;
    /* one expert at a time: unpack its three tensors, apply to its tokens */
    for (int e = 0; e < nexp && !rc; e++) {
        int shared = e == E;
        int used = shared && T > 0;
        for (int64_t a = 0; a < (int64_t)T * K && !used; a++) used = ridx[a] == e;
        if (!used) continue;
        if (oracle_unpack(fmt[3 * e + 0], (const uint8_t*)gate[e], I, H, Wg) ||
            oracle_unpack(fmt[3 * e + 1], (const uint8_t*)up[e], I, H, Wu) ||
            oracle_unpack(fmt[3 * e + 2], (const uint8_t*)down[e], H, I, Wd)) { rc = -1; break; }
        for (int t = 0; t < T; t++) {
            if (shared) {
                expert_apply(H, I, Wg, Wu, Wd, xd + (int64_t)t * H, 1.0, hbuf, yd + (int64_t)t * H);
                continue;
            }
            for (int j = 0; j < K; j++)
                if (ridx[(int64_t)t * K + j] == e)
                    expert_apply(H, I, Wg, Wu, Wd, xd + (int64_t)t * H,
                                 (double)rw[(int64_t)t * K + j], hbuf, yd + (int64_t)t * H);
        }
    }
    for (int64_t i = 0; i < (int64_t)T * H; i++) y[i] = (float)yd[i];
    if (idx) memcpy(idx, ridx, sizeof(int32_t) * (size_t)T * K);
    if (w) memcpy(w, rw, sizeof(float) * (size_t)T * K);
    free(ridx); free(rw); free(xd); free(yd); free(hbuf); free(Wg); free(Wu); free(Wd);
    return rc;
}
