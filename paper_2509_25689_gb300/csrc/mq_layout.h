// Packed-format geometry shared by the library's host codec and kernels.
// The block formats are the k-quant style types the compressed experts are
// stored in (arXiv 2509.25689 Sec. 3.3, Sec. 4.1); the byte layout is this
// library's own (documented in include/moeq.h).
#pragma once
#include <stddef.h>
#include <stdint.h>

#ifdef __CUDACC__
#define MQ_HD __host__ __device__ __forceinline__
#else
#define MQ_HD inline
#endif

namespace mq {

enum Format : int { kQ2K = 1, kQ3K = 2, kQ4K = 3, kQ80 = 4, kQ6K = 5, kBF16 = 6 };
constexpr int kNumFormats = 6;

constexpr int kPlaneAlign = 256;
constexpr int kRowTile = 32;         // records are grouped in tiles of 32 rows
constexpr int kMaxExperts = 256;     // routed experts per layer
constexpr int kMaxTopK = 32;
constexpr int kMaxGroups = 64;

MQ_HD bool valid_format(int f) { return f >= kQ2K && f <= kBF16; }

// weights per block along the contraction axis
MQ_HD int block_len(int f) { return f == kQ80 || f == kBF16 ? 32 : 256; }

// bytes per (row, block) record of each plane, planes in storage order; a
// record is stored in units of at most 64 bytes (Q4_K and Q6_K codes have 2)
struct PlaneBytes { int n; int b[4]; };
MQ_HD PlaneBytes plane_bytes(int f) {
    PlaneBytes p{0, {0, 0, 0, 0}};
    if (f == kQ4K) { p.n = 4; p.b[0] = 2; p.b[1] = 2; p.b[2] = 12; p.b[3] = 128; }
    else if (f == kQ2K) { p.n = 4; p.b[0] = 2; p.b[1] = 2; p.b[2] = 16; p.b[3] = 64; }
    else if (f == kQ3K) { p.n = 4; p.b[0] = 2; p.b[1] = 12; p.b[2] = 64; p.b[3] = 32; }
    else if (f == kQ80) { p.n = 2; p.b[0] = 2; p.b[1] = 32; }
    else if (f == kQ6K) { p.n = 4; p.b[0] = 2; p.b[1] = 16; p.b[2] = 128; p.b[3] = 64; }
    else if (f == kBF16) { p.n = 1; p.b[0] = 64; }
    return p;
}
MQ_HD int unit_bytes(int record_bytes) { return record_bytes > 64 ? 64 : record_bytes; }

MQ_HD int64_t pad_plane(int64_t v) { return (v + kPlaneAlign - 1) / kPlaneAlign * kPlaneAlign; }

// Where each plane of a [rows x cols] tensor starts, and the total size.
// Inside a plane, unit u of the record of (row r, block b) is at
//   ((((r / 32) * blocks_per_row + b) * units + u) * 32 + r % 32) * unit_bytes
// so any block range of a 32-row tile is one contiguous byte range.
struct TensorLayout {
    int64_t blocks_per_row;
    int64_t plane[4];
    int64_t total;
};

MQ_HD int64_t pad_rows(int64_t rows) { return (rows + kRowTile - 1) / kRowTile * kRowTile; }

// byte offset, from the plane start, of unit u of record (r, b)
MQ_HD int64_t unit_offset(int64_t bpr, int record_bytes, int64_t r, int64_t b, int u) {
    const int ub = unit_bytes(record_bytes), nu = record_bytes / ub;
    return ((((r / kRowTile) * bpr + b) * nu + u) * kRowTile + r % kRowTile) * ub;
}

MQ_HD TensorLayout tensor_layout(int f, int64_t rows, int64_t cols) {
    TensorLayout t{};
    const int qk = block_len(f);
    t.blocks_per_row = (cols + qk - 1) / qk;
    const int64_t nblk = pad_rows(rows) * t.blocks_per_row;
    const PlaneBytes pb = plane_bytes(f);
    int64_t at = 0;
    for (int p = 0; p < pb.n; ++p) { t.plane[p] = at; at += pad_plane(nblk * pb.b[p]); }
    for (int p = pb.n; p < 4; ++p) t.plane[p] = at;
    t.total = at;
    return t;
}

// ---- positions inside a block --------------------------------------------
// Weight k of a block lies in sub-block j = k / n (n = 16 for 2-bit and
// 1-bit codes, 32 for 4-bit and 8-bit codes), at pair m = (k % n) / 2,
// e = k % 2: the two codes of a pair sit 16 bits apart in one word, so one
// masked word is an fp16x2 MMA operand register ("pair order").
struct CodePos { int word; int bit; };

MQ_HD CodePos pos2(int k) {   // 2-bit codes: sub-block j in word 4 (j % 4) + j / 4
    const int j = k >> 4, m = (k & 15) >> 1, e = k & 1;
    return CodePos{4 * (j & 3) + (j >> 2), 16 * e + 2 * m};
}
MQ_HD CodePos pos1(int k) {   // Q3_K high-bit plane
    const int j = k >> 4, m = (k & 15) >> 1, e = k & 1;
    return CodePos{2 * (j & 3) + (j >> 3), 16 * e + 8 * ((j >> 2) & 1) + m};
}
MQ_HD CodePos pos4(int k) {   // 4-bit codes: two 64-byte units, unit = j / 4
    const int j = k >> 5, m = (k & 31) >> 1, e = k & 1;
    return CodePos{16 * (j >> 2) + 4 * (j & 3) + (m >> 2), 16 * e + 4 * (m & 3)};
}
MQ_HD CodePos pos8(int k) {   // Q8_0 codes (stored q + 128), k < 32
    const int m = k >> 1, e = k & 1;
    return CodePos{m >> 1, 16 * e + 8 * (m & 1)};
}
// Q6_K low nibbles (16-wide sub-blocks): two 64-byte units, unit = j / 8;
// sub-block j in words 16 (j / 8) + 4 (j % 4) + 2 ((j / 4) % 2) + 0..1
MQ_HD CodePos pos4s(int k) {
    const int j = k >> 4, m = (k & 15) >> 1, e = k & 1;
    return CodePos{16 * (j >> 3) + 4 * (j & 3) + 2 * ((j >> 2) & 1) + (m >> 2), 16 * e + 4 * (m & 3)};
}
// BF16 block of 32: 16-bit position of weight k (tensor-core fragment order:
// the words for k = 2t, 2t+1 | 8+2t, 9+2t | 16+2t, 17+2t | 24+2t, 25+2t
// are contiguous)
MQ_HD int bf16_slot(int k) { return 8 * ((k & 7) >> 1) + 2 * (k >> 3) + (k & 1); }

// slot of sub-block j (< 16) in the Q2_K / Q3_K scale fields
MQ_HD int q16_slot(int j) { return 4 * ((j & 7) >> 1) + 2 * (j >> 3) + (j & 1); }

MQ_HD uint32_t load_le32(const uint8_t* p) {
    return (uint32_t)p[0] | ((uint32_t)p[1] << 8) | ((uint32_t)p[2] << 16) | ((uint32_t)p[3] << 24);
}
MQ_HD uint16_t load_le16(const uint8_t* p) { return (uint16_t)(p[0] | (p[1] << 8)); }

// Q3_K stored 6-bit scale of sub-block j
MQ_HD int q3_scale_field(const uint8_t* s, int j) {
    const int u = q16_slot(j);
    const int lo = (s[u >> 1] >> ((u & 1) * 4)) & 15;
    const int hi = (s[8 + (u >> 2)] >> ((u & 3) * 2)) & 3;
    return lo | (hi << 4);
}

// Q4_K 6-bit sub-scale and sub-min of sub-block j (< 8)
MQ_HD void q4_fields(const uint8_t* s, int j, int& sc, int& m) {
    const uint32_t high = load_le32(s + 8) >> (4 * j);
    sc = (s[j] & 15) | (int)((high & 3u) << 4);
    m = (s[j] >> 4) | (int)(((high >> 2) & 3u) << 4);
}

// exact fp16 -> fp32 (library's own conversion)
MQ_HD float half_bits_to_float(uint16_t h) {
    const uint32_t s = (uint32_t)(h >> 15) << 31;
    const uint32_t ex = (h >> 10) & 31u, mt = h & 1023u;
    uint32_t bits;
    if (ex == 31u) bits = s | 0x7f800000u | (mt << 13);
    else if (ex != 0u) bits = s | ((ex + 112u) << 23) | (mt << 13);
    else {
        // subnormal / zero: mt * 2^-24 (exact)
        float v = (float)mt * 5.9604644775390625e-08f;
        return s ? -v : v;
    }
    union { uint32_t u; float f; } c; c.u = bits; return c.f;
}

// Scalar dequantization of weight (row r, column c) of a packed tensor.
// Slow reference-style access used by the device unpack kernel and the host
// codec.
MQ_HD uint32_t rec_word(const uint8_t* plane, const TensorLayout& L, int rb, int64_t r, int64_t b, int word) {
    const int ub = unit_bytes(rb);
    const int u = (4 * word) / ub;
    return load_le32(plane + unit_offset(L.blocks_per_row, rb, r, b, u) + (4 * word) % ub);
}
MQ_HD const uint8_t* rec_ptr(const uint8_t* plane, const TensorLayout& L, int rb, int64_t r, int64_t b) {
    return plane + unit_offset(L.blocks_per_row, rb, r, b, 0);
}

MQ_HD float dequant_at(int f, const uint8_t* base, const TensorLayout& L, int64_t r, int64_t c) {
    const int qk = block_len(f);
    const int64_t b = c / qk;
    const int k = (int)(c % qk);
    const PlaneBytes pb = plane_bytes(f);
    if (f == kBF16) {
        const uint16_t h = load_le16(rec_ptr(base + L.plane[0], L, 64, r, b) + 2 * bf16_slot(k));
        union { uint32_t u; float f; } c; c.u = (uint32_t)h << 16; return c.f;
    }
    if (f == kQ6K) {
        const float d = half_bits_to_float(load_le16(rec_ptr(base + L.plane[0], L, 2, r, b)));
        const int s = (int)rec_ptr(base + L.plane[1], L, 16, r, b)[q16_slot(k >> 4)] - 128;
        const CodePos pl = pos4s(k), ph = pos2(k);
        const int lo = (int)((rec_word(base + L.plane[2], L, 128, r, b, pl.word) >> pl.bit) & 15u);
        const int hi = (int)((rec_word(base + L.plane[3], L, 64, r, b, ph.word) >> ph.bit) & 3u);
        return (d * (float)s) * (float)((lo | (hi << 4)) - 32);
    }
    const float d = half_bits_to_float(load_le16(rec_ptr(base + L.plane[0], L, 2, r, b)));
    if (f == kQ80) {
        const CodePos p = pos8(k);
        const int q = (int)((rec_word(base + L.plane[1], L, 32, r, b, p.word) >> p.bit) & 0xffu) - 128;
        return d * (float)q;
    }
    if (f == kQ3K) {
        const int s = q3_scale_field(rec_ptr(base + L.plane[1], L, 12, r, b), k >> 4);
        const CodePos pl = pos2(k), ph = pos1(k);
        const int lo = (int)((rec_word(base + L.plane[2], L, 64, r, b, pl.word) >> pl.bit) & 3u);
        const int hi = (int)((rec_word(base + L.plane[3], L, 32, r, b, ph.word) >> ph.bit) & 1u);
        return (d * (float)(s - 32)) * (float)((lo | (hi << 2)) - 4);
    }
    const float dm = half_bits_to_float(load_le16(rec_ptr(base + L.plane[1], L, 2, r, b)));
    int sc, m, q;
    if (f == kQ4K) {
        q4_fields(rec_ptr(base + L.plane[2], L, 12, r, b), k >> 5, sc, m);
        const CodePos p = pos4(k);
        q = (int)((rec_word(base + L.plane[3], L, pb.b[3], r, b, p.word) >> p.bit) & 15u);
    } else {
        const uint8_t bt = rec_ptr(base + L.plane[2], L, 16, r, b)[q16_slot(k >> 4)];
        sc = bt & 15; m = bt >> 4;
        const CodePos p = pos2(k);
        q = (int)((rec_word(base + L.plane[3], L, 64, r, b, p.word) >> p.bit) & 3u);
    }
    // (d*sc)*q is exact; the subtraction is the only rounding (FMA-invariant)
    return (d * (float)sc) * (float)q - dm * (float)m;
}

}  // namespace mq
