// Philox4x32-10 and the exact fp32 decision of Eq. 9, shared by the
// per-parameter select kernels and the per-message decision kernel.
#pragma once

#include <stdint.h>

namespace fasgd {

// Philox4x32-10 (Salmon, Moraes, Dror, Shaw, SC'11): ten rounds, each two
// 32x32->64 products of the counter's even words with the round multipliers,
// the high halves xor-ed with the odd words and the round key.  The key
// schedule (seed advanced by the Weyl constants) is precomputed on the host.
// Each product is formed as separate high and low 32-bit multiplies (the same
// bits as one widening multiply; measured 0.5-0.9 us faster per 25M select).
constexpr uint32_t kPhiloxM0 = 0xD2511F53u, kPhiloxM1 = 0xCD9E8D57u;
constexpr uint32_t kPhiloxW0 = 0x9E3779B9u, kPhiloxW1 = 0xBB67AE85u;

inline void philox_key_schedule(uint64_t seed, uint32_t rk0[10], uint32_t rk1[10]) {
    uint32_t k0 = (uint32_t)seed, k1 = (uint32_t)(seed >> 32);
    for (int r = 0; r < 10; ++r) {
        rk0[r] = k0;
        rk1[r] = k1;
        k0 += kPhiloxW0;
        k1 += kPhiloxW1;
    }
}

struct Philox4 {
    uint32_t x[4];
};

__device__ __forceinline__ Philox4 philox4x32_10(uint32_t c0, uint32_t c1, uint32_t c2,
                                                 uint32_t c3, const uint32_t (&rk0)[10],
                                                 const uint32_t (&rk1)[10]) {
#pragma unroll
    for (int r = 0; r < 10; ++r) {
        const uint32_t hi0 = __umulhi(kPhiloxM0, c0), lo0 = kPhiloxM0 * c0;
        const uint32_t hi1 = __umulhi(kPhiloxM1, c2), lo1 = kPhiloxM1 * c2;
        c0 = hi1 ^ c1 ^ rk0[r];
        c1 = lo1;
        c2 = hi0 ^ c3 ^ rk1[r];
        c3 = lo0;
    }
    Philox4 o;
    o.x[0] = c0;
    o.x[1] = c1;
    o.x[2] = c2;
    o.x[3] = c3;
    return o;
}

// Eq. 9 for one parameter: send iff u / 2^24 < 1 / (1 + c / a), a = fl(v + eps_b),
// i.e. iff u * d < a * 2^24 with d = fl(a + c), decided exactly.
//
// The sign of u * d - a * 2^24 is the sign of one fused multiply-add: it
// rounds the exact value once, rounding keeps the sign, and a nonzero
// difference of these operands (all multiples of 2^-149) is never rounded to
// zero.  So the test is fma(u, d, -A) < 0 with A = a * 2^24, once A is exact.
// Two scalings cover every a >= 0 and c >= 0 (+inf included):
//   SCALE_D = false, for c < kSendScaleC = 2^79:  fma(u, d, -(a * 2^24)).
//     A is exact below a = 2^104; from there on d = a (c is below half an
//     ulp of a), where u < 2^24 always holds, and the overflowed A = +inf
//     still gives fma = -inf < 0.
//   SCALE_D = true, for c >= 2^79:  fma(u, d * 2^-24, -a).  d >= c >= 2^79,
//     so d * 2^-24 is exact; d = +inf gives +inf (u > 0) or NaN (u = 0),
//     neither below 0: nothing is sent, as Eq. 9 says for c = +inf.
// The host picks the form once per call from c (send_form).
constexpr float kSendScaleC = 604462909807314587353088.0f;  // 2^79

inline bool send_form(float c) { return c >= kSendScaleC; }

template <bool SCALE_D>
__device__ __forceinline__ bool send_test(uint32_t u, float v, float c, float eps_b) {
    const float a = __fadd_rn(v, eps_b);
    const float d = __fadd_rn(a, c);
    const float uf = (float)u;  // exact: u < 2^24
    const float s = SCALE_D ? __fmaf_rn(uf, __fmul_rn(d, 5.9604644775390625e-8f), -a)
                            : __fmaf_rn(uf, d, -__fmul_rn(a, 16777216.0f));
    return s < 0.0f;
}

// The same test with the form chosen per call (single decisions).
__device__ __forceinline__ uint32_t send_bit(uint32_t u, float v, float c, float eps_b) {
    return (c >= kSendScaleC ? send_test<true>(u, v, c, eps_b) : send_test<false>(u, v, c, eps_b))
               ? 1u : 0u;
}

}  // namespace fasgd
