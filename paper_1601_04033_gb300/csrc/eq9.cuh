// Philox4x32-10 and the exact fp32 decision of Eq. 9, shared by the
// per-parameter select kernels and the per-message decision kernel.
#pragma once

#include <stdint.h>

namespace fasgd {

// Philox4x32-10 (Salmon, Moraes, Dror, Shaw, SC'11): ten rounds, each two
// 32x32->64 products of the counter's even words with the round multipliers,
// the high halves xor-ed with the odd words and the round key.  The key
// schedule (seed advanced by the Weyl constants) is precomputed on the host.
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
        const uint64_t p0 = (uint64_t)kPhiloxM0 * c0;
        const uint64_t p1 = (uint64_t)kPhiloxM1 * c2;
        c0 = (uint32_t)(p1 >> 32) ^ c1 ^ rk0[r];
        c1 = (uint32_t)p1;
        c2 = (uint32_t)(p0 >> 32) ^ c3 ^ rk1[r];
        c3 = (uint32_t)p0;
    }
    Philox4 o;
    o.x[0] = c0;
    o.x[1] = c1;
    o.x[2] = c2;
    o.x[3] = c3;
    return o;
}

// Eq. 9 for one parameter: send iff u / 2^24 < 1 / (1 + c / a), a = fl(v + eps_b),
// i.e. iff u * d < A with d = fl(a + c) and A = a * 2^24, decided exactly:
// u * d = prod + err exactly (prod = fl(u * d), err = fma(u, d, -prod)), and
// u * d < A  <=>  err < A - prod  <=>  err < fl(A - prod).  The last step is
// exact: when A and prod are within a factor of two, A - prod is exact
// (Sterbenz); otherwise |A - prod| > 2^-24 prod >= |err|, and rounding
// A - prod keeps it on the same side of err.
__device__ __forceinline__ uint32_t send_bit(uint32_t u, float v, float c, float eps_b) {
    const float a = __fadd_rn(v, eps_b);
    const float d = __fadd_rn(a, c);
    const float uf = (float)u;  // exact: u < 2^24
    const float prod = __fmul_rn(uf, d);
    const float err = __fmaf_rn(uf, d, -prod);
    const float A = __fmul_rn(a, 16777216.0f);
    return err < __fsub_rn(A, prod) ? 1u : 0u;
}

}  // namespace fasgd
