// Portable four-lane e^x for the host-side block (softmax and SiLU of the CPU suffix), in GCC
// vector extensions only, so the same source builds for NEON (Arm) and SSE (x86) lanes.
//
// Method (Cody and Waite's argument reduction, then a polynomial): x = n ln2 + r with
// n = round(x log2 e), r = x - n c1 - n c2, where c1 = 355/512 holds the leading 9 bits of
// ln 2 (so n c1 is exact for |n| <= 2^15) and c2 = ln 2 - c1 rounded to fp32; |r| <= ln2/2
// up to rounding. e^r is the Taylor series of e^r to degree 7 in Horner form: its
// truncation error is below r^8/8! < 5.3e-9 relative on that interval, under the fp32
// rounding of the evaluation itself. The result is e^r times 2^n, the latter written straight
// into the exponent field.
//
// Range: x <= -87.33 (below ln of the smallest normal fp32, including -inf) gives 0, so
// results that would be subnormal are flushed; x >= 88.72 (above ln of the largest fp32)
// gives +inf. NaN is not an input of the callers (softmax arguments s - max(s) and SiLU's
// -g of finite g).
#pragma once

#include <cstdint>
#include <cstring>

namespace vla_cpu {

typedef float v4f __attribute__((vector_size(16)));
typedef int32_t v4i __attribute__((vector_size(16)));

inline v4f exp4(v4f x) {
    const float kLog2e = 1.4426950408889634f;
    const float kShift = 12582912.0f;  // 1.5 * 2^23: adding and subtracting it rounds to an integer
    const float kC1 = 0.693359375f;    // 355 / 512
    const float kC2 = -2.12194440e-4f; // ln 2 - 355/512
    const float kLo = -87.3365479f;    // ln(2^-126)
    const float kHi = 88.7228394f;     // ln of the largest finite fp32
    const v4i under = x < kLo;
    const v4i over = x > kHi;
    x = x < kLo ? (v4f){kLo, kLo, kLo, kLo} : x;
    x = x > kHi ? (v4f){kHi, kHi, kHi, kHi} : x;
    const v4f n = (x * kLog2e + kShift) - kShift;
    v4f r = x - n * kC1;
    r = r - n * kC2;
    v4f p = r * (1.0f / 5040.0f) + (1.0f / 720.0f);
    p = p * r + (1.0f / 120.0f);
    p = p * r + (1.0f / 24.0f);
    p = p * r + (1.0f / 6.0f);
    p = p * r + 0.5f;
    p = p * r + 1.0f;
    p = p * r + 1.0f;
    // 2^n in two halves so that n = 128 (x near the top of the range) stays representable
    const v4i ni = __builtin_convertvector(n, v4i);
    const v4i h1 = ni >> 1, h2 = ni - h1;
    const v4i b1 = (h1 + 127) << 23, b2 = (h2 + 127) << 23;
    v4f s1, s2;
    std::memcpy(&s1, &b1, sizeof s1);
    std::memcpy(&s2, &b2, sizeof s2);
    v4f y = (p * s1) * s2;
    v4i yb;
    std::memcpy(&yb, &y, sizeof yb);
    const v4i inf_bits = {0x7F800000, 0x7F800000, 0x7F800000, 0x7F800000};
    yb = (yb & ~under & ~over) | (inf_bits & over);
    std::memcpy(&y, &yb, sizeof y);
    return y;
}

inline float exp1(float x) {
    const v4f v = {x, x, x, x};
    return exp4(v)[0];
}

}  // namespace vla_cpu
