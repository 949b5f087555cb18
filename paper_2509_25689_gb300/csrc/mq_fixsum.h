// Order-free sums of routing weights for the expert-importance score (arXiv
// 2509.25689 Sec. 3.1: s_e, the mean routing weight of expert e's
// selections).  A weight is rounded to the nearest multiple of 2^-64 (ties
// to even; exact for every float32 with |w| >= 2^-40) and held as a signed
// 128-bit integer count of 2^-64 units in two 64-bit words (two's
// complement, hi:lo).  Integer addition is associative, so the sum has the
// same bits in any order; the total is rounded once to double.  Shared by
// the host routine and the device histogram.
#pragma once
#include <math.h>
#include <cstdint>
#include <cstring>

#if defined(__CUDACC__)
#define MQ_FIX_HD __host__ __device__ __forceinline__
#else
#define MQ_FIX_HD inline
#endif

namespace mq {

struct Fix128 {
    uint64_t lo, hi;
};

// Weights must be finite with |w| < 2^32 (so that 2^31 of them cannot
// overflow the 63-bit integer part); returns false otherwise.
MQ_FIX_HD bool fix_from_float(float w, Fix128& out) {
    uint32_t u;
#if defined(__CUDA_ARCH__)
    u = __float_as_uint(w);
#else
    std::memcpy(&u, &w, 4);
#endif
    const uint32_t ex = (u >> 23) & 0xFFu;
    const bool neg = (u >> 31) != 0;
    if (ex == 0xFFu || ex >= 127u + 32u) return false;
    uint64_t lo = 0, hi = 0;
    if (ex != 0) {   // subnormals are below 2^-126: they round to 0 units
        const uint32_t m = (u & 0x7FFFFFu) | 0x800000u;   // w = m * 2^(ex - 150) = m * 2^(ex - 86) units
        if (ex >= 86u) {
            const uint32_t s = ex - 86u;                   // 0..72
            if (s < 64u) {
                lo = (uint64_t)m << s;
                hi = s == 0 ? 0 : (uint64_t)m >> (64u - s);
            } else {
                hi = (uint64_t)m << (s - 64u);
            }
        } else {
            const uint32_t s = 86u - ex;                   // 1..85
            if (s <= 24u) {                                // m < 2^24: beyond 24 the quotient is < 1/2
                uint32_t q = m >> s;
                const uint32_t r = m & ((1u << s) - 1u), half = 1u << (s - 1u);
                if (r > half || (r == half && (q & 1u))) ++q;
                lo = q;
            }
        }
    }
    if (neg) {   // two's complement negation
        lo = ~lo + 1u;
        hi = ~hi + (lo == 0 ? 1u : 0u);
    }
    out.lo = lo;
    out.hi = hi;
    return true;
}

// The 128-bit sum rounded to the nearest double (ties to even), times 2^-64.
MQ_FIX_HD double fix_to_double(Fix128 v) {
    const bool neg = (v.hi >> 63) != 0;
    uint64_t lo = v.lo, hi = v.hi;
    if (neg) {
        lo = ~lo + 1u;
        hi = ~hi + (lo == 0 ? 1u : 0u);
    }
    if (hi == 0 && lo < (1ull << 53)) {
        const double r = ldexp((double)lo, -64);
        return neg ? -r : r;
    }
    // top bit position p >= 53; keep 53 bits
    int p = 0;
    if (hi != 0) {
        for (int b = 63; b >= 0; --b)
            if ((hi >> b) & 1u) { p = 64 + b; break; }
    } else {
        for (int b = 63; b >= 0; --b)
            if ((lo >> b) & 1u) { p = b; break; }
    }
    const int sh = p - 52;   // 1..75
    uint64_t mant, rem_hi, rem_lo;   // mant = v >> sh; rem = v mod 2^sh
    if (sh < 64) {
        mant = (lo >> sh) | (hi << (64 - sh));
        rem_hi = 0;
        rem_lo = lo & ((1ull << sh) - 1u);
    } else {
        mant = hi >> (sh - 64);
        rem_hi = sh == 64 ? 0 : hi & ((1ull << (sh - 64)) - 1u);
        rem_lo = lo;
    }
    // half = 2^(sh - 1)
    const uint64_t half_hi = sh - 1 >= 64 ? 1ull << (sh - 1 - 64) : 0;
    const uint64_t half_lo = sh - 1 >= 64 ? 0 : 1ull << (sh - 1);
    const bool above = rem_hi > half_hi || (rem_hi == half_hi && rem_lo > half_lo);
    const bool tie = rem_hi == half_hi && rem_lo == half_lo;
    if (above || (tie && (mant & 1u))) ++mant;   // mant <= 2^53: exact in a double
    const double r = ldexp((double)mant, sh - 64);
    return neg ? -r : r;
}

MQ_FIX_HD void fix_add(Fix128& acc, Fix128 v) {
    const uint64_t lo = acc.lo + v.lo;
    acc.hi += v.hi + (lo < acc.lo ? 1u : 0u);
    acc.lo = lo;
}

}  // namespace mq
