// Per-element server update rules, shared by the dense and sparse kernels.
#pragma once

#include "kernels.cuh"

namespace fasgd {

// Hardware approximations (PTX rsqrt.approx.f32 / rcp.approx.f32, subnormals
// kept).  Their error is a few ulp, far inside the 1e-5 relative bound the
// results are held to; see the rounding notes on fasgd_update below.
__device__ __forceinline__ float rsqrt_approx(float x) {
    float y;
    asm("rsqrt.approx.f32 %0, %1;" : "=f"(y) : "f"(x));
    return y;
}

__device__ __forceinline__ float rcp_approx(float x) {
    float y;
    asm("rcp.approx.f32 %0, %1;" : "=f"(y) : "f"(x));
    return y;
}

// ASGD / SASGD (Eq. 1-2): theta <- theta - alpha(tau) * g.  Both operations
// are rounded separately (no fused multiply-add), so the result is the
// correctly rounded fp32 sequence.
__device__ __forceinline__ void sgd_update(float& theta, float g, float coef) {
    theta = __fsub_rn(theta, __fmul_rn(coef, g));
}

// FASGD (Eq. 4-8) for one parameter and one gradient entry g.
//   Eq. 4  n <- gamma n + (1 - gamma) g^2
//   Eq. 5  b <- gamma b + (1 - gamma) g
//   Eq. 6  v <- beta v + (1 - beta) / sqrt(max(n - b^2, 0) + eps)
//   Eq. 7-8 theta <- theta - alpha(tau) * g / v      (v just updated)
// n, b and the radicand are formed with one rounding per product and sum
// (no contraction), which makes them the exact fp32 sequence.  The inverse
// square root, the reciprocal of v and the two fused multiply-adds of the
// v and theta updates differ from a once-rounded sequence by a few ulp; v is
// a positive weighted mean, so that difference does not grow, and theta only
// accumulates it relative to the size of each step.
__device__ __forceinline__ void fasgd_update(float& theta, float& n, float& b, float& v,
                                             float g, float coef, const StatParams& sp) {
    n = __fadd_rn(__fmul_rn(sp.gamma, n), __fmul_rn(sp.one_m_gamma, __fmul_rn(g, g)));
    b = __fadd_rn(__fmul_rn(sp.gamma, b), __fmul_rn(sp.one_m_gamma, g));
    const float var = fmaxf(__fsub_rn(n, __fmul_rn(b, b)), 0.0f);
    const float r = rsqrt_approx(__fadd_rn(var, sp.eps));
    v = fmaf(sp.beta, v, sp.one_m_beta * r);
    theta = fmaf(-(coef * g), rcp_approx(v), theta);
}

}  // namespace fasgd
