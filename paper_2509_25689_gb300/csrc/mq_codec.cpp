// Host codec: quantizer (pack) and dequantizer (unpack) for the block
// formats of include/moeq.h.  The paper quantizes each tensor to a llama.cpp
// style block type (arXiv 2509.25689 Sec. 3.3); the rule here is this
// library's deterministic nearest-grid quantizer:
//   asymmetric (Q4_K L=15 S=63, Q2_K L=3 S=15), per sub-block j:
//     lo = min(0, min w), hi = max w, scale = (hi-lo)/L, mn = -lo
//     d = fp16(max scale / S), dmin = fp16(max mn / S)
//     sc = clamp(rne(scale/d), 0, S), m = clamp(rne(mn/dmin), 0, S)
//     q  = clamp(rne((w + dmin*m) / (d*sc)), 0, L)
//   Q3_K: a = sub-block weight of largest |w| (first), scale = a / -4,
//     d = fp16(max |scale| / 31), sc = clamp(rne(scale/d), -32, 31),
//     q = clamp(rne(w / (d*sc)), -4, 3); stored sc+32 and q+4
//   Q8_0: d = fp16(max|w| / 127), q = clamp(rne(w/d), -127, 127), stored q+128
//   Q6_K: as Q3_K with codes -32..31 and 8-bit scales: scale = a / -32,
//     d = fp16(max |scale| / 127), sc = clamp(rne(scale/d), -128, 127),
//     q = clamp(rne(w / (d*sc)), -32, 31); stored sc+128 and q+32
//   BF16: each weight rounded to bf16 (nearest, ties to even); a weight that
//     rounds past the largest finite bf16 is rejected
// All arithmetic is IEEE fp32 (this file is built with -ffp-contract=off),
// rne = round half to even; a zero denominator gives code 0.
#include <cmath>
#include <cstring>
#include <vector>

#include "../../include/moeq.h"
#include "mq_layout.h"

namespace {

using namespace mq;

uint16_t to_half_rne(float f) {
    uint32_t u;
    std::memcpy(&u, &f, 4);
    const uint16_t sign = (uint16_t)((u >> 16) & 0x8000u);
    const uint32_t a = u & 0x7fffffffu;
    if (a > 0x7f800000u) return (uint16_t)(sign | 0x7e00u);
    if (a >= 0x38800000u) {  // normal fp16 range (or overflow)
        const uint32_t r = a - 0x38000000u;
        uint32_t h = (r + 0x0fffu + ((r >> 13) & 1u)) >> 13;
        if (h > 0x7c00u) h = 0x7c00u;
        return (uint16_t)(sign | h);
    }
    // subnormal: integer multiple of 2^-24, scaling by 2^24 is exact
    const float v = std::fabs(f) * 16777216.0f;
    return (uint16_t)(sign | (uint16_t)std::nearbyint(v));
}

int rne(float v) { return (int)std::nearbyint(v); }
int clip(int v, int lo, int hi) { return v < lo ? lo : (v > hi ? hi : v); }

void store16(uint8_t* p, uint16_t v) { p[0] = (uint8_t)(v & 0xff); p[1] = (uint8_t)(v >> 8); }

void set_bits(uint8_t* words, CodePos p, uint32_t v, uint32_t mask) {
    uint32_t w = load_le32(words + 4 * p.word);
    w = (w & ~(mask << p.bit)) | ((v & mask) << p.bit);
    for (int b = 0; b < 4; ++b) words[4 * p.word + b] = (uint8_t)(w >> (8 * b));
}

struct AsymBlock { uint16_t d, dmin; int sc[16], m[16], q[256]; };

void quantize_asym(const float* w, int sub, int L, int S, AsymBlock& out) {
    const int nsub = 256 / sub;
    float scale[16], mn[16];
    float top_scale = 0.0f, top_mn = 0.0f;
    for (int j = 0; j < nsub; ++j) {
        const float* v = w + j * sub;
        float lo = 0.0f, hi = v[0];
        for (int i = 0; i < sub; ++i) { lo = v[i] < lo ? v[i] : lo; hi = v[i] > hi ? v[i] : hi; }
        scale[j] = (hi - lo) / (float)L;
        mn[j] = 0.0f - lo;
        top_scale = scale[j] > top_scale ? scale[j] : top_scale;
        top_mn = mn[j] > top_mn ? mn[j] : top_mn;
    }
    out.d = to_half_rne(top_scale / (float)S);
    out.dmin = to_half_rne(top_mn / (float)S);
    const float d = half_bits_to_float(out.d), dmin = half_bits_to_float(out.dmin);
    for (int j = 0; j < nsub; ++j) {
        out.sc[j] = d > 0.0f ? clip(rne(scale[j] / d), 0, S) : 0;
        out.m[j] = dmin > 0.0f ? clip(rne(mn[j] / dmin), 0, S) : 0;
        const float den = d * (float)out.sc[j];
        const float shift = dmin * (float)out.m[j];
        for (int i = 0; i < sub; ++i) {
            const float num = w[j * sub + i] + shift;
            out.q[j * sub + i] = den > 0.0f ? clip(rne(num / den), 0, L) : 0;
        }
    }
}

// bf16 of a finite float, nearest-even; false if it rounds to infinity
bool to_bf16_rne(float f, uint16_t& out) {
    uint32_t u;
    std::memcpy(&u, &f, 4);
    const uint32_t low = u & 0xffffu, keep = u >> 16;
    const bool up = low > 0x8000u || (low == 0x8000u && (keep & 1u));
    const uint32_t h = keep + (up ? 1u : 0u);
    out = (uint16_t)h;
    return ((h >> 7) & 0xffu) != 0xffu;
}

void encode_block(int f, const float* w, uint8_t* const planes[4]) {
    if (f == kBF16) {
        for (int k = 0; k < 32; ++k) {
            uint16_t h = 0;
            to_bf16_rne(w[k], h);   // range checked before encoding
            store16(planes[0] + 2 * bf16_slot(k), h);
        }
        return;
    }
    if (f == kQ6K) {
        float scale[16], top = 0.0f;
        for (int j = 0; j < 16; ++j) {
            float a = w[16 * j];
            for (int i = 1; i < 16; ++i) if (std::fabs(w[16 * j + i]) > std::fabs(a)) a = w[16 * j + i];
            scale[j] = a / -32.0f;
            top = std::fabs(scale[j]) > top ? std::fabs(scale[j]) : top;
        }
        const uint16_t dh = to_half_rne(top / 127.0f);
        const float d = half_bits_to_float(dh);
        store16(planes[0], dh);
        for (int j = 0; j < 16; ++j) {
            const int sc = d > 0.0f ? clip(rne(scale[j] / d), -128, 127) : 0;
            planes[1][q16_slot(j)] = (uint8_t)(sc + 128);
            const float den = d * (float)sc;
            for (int i = 0; i < 16; ++i) {
                const int k = 16 * j + i;
                const int q = (den != 0.0f ? clip(rne(w[k] / den), -32, 31) : 0) + 32;
                set_bits(planes[2], pos4s(k), (uint32_t)q, 15u);
                set_bits(planes[3], pos2(k), (uint32_t)(q >> 4), 3u);
            }
        }
        return;
    }
    if (f == kQ80) {
        float amax = 0.0f;
        for (int k = 0; k < 32; ++k) amax = std::fabs(w[k]) > amax ? std::fabs(w[k]) : amax;
        const uint16_t dh = to_half_rne(amax / 127.0f);
        const float d = half_bits_to_float(dh);
        store16(planes[0], dh);
        for (int k = 0; k < 32; ++k) {
            const int q = d > 0.0f ? clip(rne(w[k] / d), -127, 127) : 0;
            set_bits(planes[1], pos8(k), (uint32_t)(q + 128), 0xffu);
        }
        return;
    }
    if (f == kQ3K) {
        float scale[16], top = 0.0f;
        for (int j = 0; j < 16; ++j) {
            float a = w[16 * j];
            for (int i = 1; i < 16; ++i) if (std::fabs(w[16 * j + i]) > std::fabs(a)) a = w[16 * j + i];
            scale[j] = a / -4.0f;
            top = std::fabs(scale[j]) > top ? std::fabs(scale[j]) : top;
        }
        const uint16_t dh = to_half_rne(top / 31.0f);
        const float d = half_bits_to_float(dh);
        store16(planes[0], dh);
        for (int j = 0; j < 16; ++j) {
            const int sc = d > 0.0f ? clip(rne(scale[j] / d), -32, 31) : 0;
            const int s = sc + 32, u = q16_slot(j);
            planes[1][u >> 1] = (uint8_t)((planes[1][u >> 1] & ~(0xf << (4 * (u & 1)))) | ((s & 15) << (4 * (u & 1))));
            planes[1][8 + (u >> 2)] = (uint8_t)((planes[1][8 + (u >> 2)] & ~(3 << (2 * (u & 3)))) |
                                                (((s >> 4) & 3) << (2 * (u & 3))));
            const float den = d * (float)sc;
            for (int i = 0; i < 16; ++i) {
                const int k = 16 * j + i;
                const int q = (den != 0.0f ? clip(rne(w[k] / den), -4, 3) : 0) + 4;
                set_bits(planes[2], pos2(k), (uint32_t)q, 3u);
                set_bits(planes[3], pos1(k), (uint32_t)(q >> 2), 1u);
            }
        }
        return;
    }
    AsymBlock b;
    const bool q4 = f == kQ4K;
    quantize_asym(w, q4 ? 32 : 16, q4 ? 15 : 3, q4 ? 63 : 15, b);
    store16(planes[0], b.d);
    store16(planes[1], b.dmin);
    if (q4) {
        uint32_t high = 0;
        for (int j = 0; j < 8; ++j) {
            planes[2][j] = (uint8_t)((b.sc[j] & 15) | ((b.m[j] & 15) << 4));
            high |= (uint32_t)((b.sc[j] >> 4) & 3) << (4 * j);
            high |= (uint32_t)((b.m[j] >> 4) & 3) << (4 * j + 2);
        }
        for (int i = 0; i < 4; ++i) planes[2][8 + i] = (uint8_t)(high >> (8 * i));
        for (int k = 0; k < 256; ++k) set_bits(planes[3], pos4(k), (uint32_t)b.q[k], 15u);
    } else {
        for (int j = 0; j < 16; ++j) planes[2][q16_slot(j)] = (uint8_t)(b.sc[j] | (b.m[j] << 4));
        for (int k = 0; k < 256; ++k) set_bits(planes[3], pos2(k), (uint32_t)b.q[k], 3u);
    }
}

}  // namespace

extern "C" size_t mq_packed_size(int fmt, int64_t rows, int64_t cols) {
    if (!valid_format(fmt) || rows < 0 || cols < 0) return 0;
    return (size_t)tensor_layout(fmt, rows, cols).total;
}

extern "C" int mq_pack(int fmt, const float* w, int64_t rows, int64_t cols, void* dst, size_t dst_bytes) {
    if (!valid_format(fmt)) return MQ_EFORMAT;
    if (rows < 0 || cols < 0 || !dst || (rows * cols > 0 && !w)) return MQ_EINVAL;
    const TensorLayout L = tensor_layout(fmt, rows, cols);
    if (dst_bytes < (size_t)L.total) return MQ_EINVAL;
    for (int64_t i = 0; i < rows * cols; ++i) {
        if (!std::isfinite(w[i])) return MQ_EINVAL;
        uint16_t h;
        if (fmt == kBF16 && !to_bf16_rne(w[i], h)) return MQ_EINVAL;
    }
    uint8_t* out = static_cast<uint8_t*>(dst);
    std::memset(out, 0, (size_t)L.total);
    const int qk = block_len(fmt);
    const PlaneBytes pb = plane_bytes(fmt);
    std::vector<float> blk(qk);
    uint8_t rec[4][128];
    // rows past `rows` (up to the 32-row tile) are encoded as zero rows
    for (int64_t r = 0; r < pad_rows(rows); ++r) {
        for (int64_t b = 0; b < L.blocks_per_row; ++b) {
            for (int k = 0; k < qk; ++k) {
                const int64_t c = b * qk + k;
                blk[k] = (r < rows && c < cols) ? w[r * cols + c] : 0.0f;
            }
            std::memset(rec, 0, sizeof(rec));
            uint8_t* planes[4] = {rec[0], rec[1], rec[2], rec[3]};
            encode_block(fmt, blk.data(), planes);
            for (int p = 0; p < pb.n; ++p) {
                const int ub = unit_bytes(pb.b[p]);
                for (int u = 0; u < pb.b[p] / ub; ++u)
                    std::memcpy(out + L.plane[p] + unit_offset(L.blocks_per_row, pb.b[p], r, b, u), rec[p] + u * ub,
                                (size_t)ub);
            }
        }
    }
    return MQ_OK;
}

extern "C" int mq_unpack(int fmt, const void* src, int64_t rows, int64_t cols, float* dst) {
    if (!valid_format(fmt)) return MQ_EFORMAT;
    if (rows < 0 || cols < 0 || (rows * cols > 0 && (!src || !dst))) return MQ_EINVAL;
    const TensorLayout L = tensor_layout(fmt, rows, cols);
    const uint8_t* in = static_cast<const uint8_t*>(src);
    for (int64_t r = 0; r < rows; ++r)
        for (int64_t c = 0; c < cols; ++c) dst[r * cols + c] = dequant_at(fmt, in, L, r, c);
    return MQ_OK;
}
