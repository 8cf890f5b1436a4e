// Per-element server update rules, shared by the dense and sparse kernels.
#pragma once

#include "kernels.cuh"

namespace fasgd {

// Hardware approximations (PTX rsqrt.approx / rcp.approx).  Their error is a
// few ulp, far inside the 1e-5 relative bound the results are held to; see
// the rounding notes on fasgd_update below.  FTZ selects the forms that flush
// subnormal inputs and outputs to zero.  In fasgd_update they give the same
// results as the subnormal-preserving forms whenever eps >= 2^-126 and the
// gradients are finite: the radicand is then at least 2^-126, and v, a
// weighted mean of r >= (1 - beta) / sqrt(FLT_MAX) with 1 - beta >= 2^-24,
// is at least 2^-88; neither they nor their reciprocals are subnormal.
template <bool FTZ>
__device__ __forceinline__ float rsqrt_approx(float x) {
    float y;
    if (FTZ)
        asm("rsqrt.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
    else
        asm("rsqrt.approx.f32 %0, %1;" : "=f"(y) : "f"(x));
    return y;
}

template <bool FTZ>
__device__ __forceinline__ float rcp_approx(float x) {
    float y;
    if (FTZ)
        asm("rcp.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
    else
        asm("rcp.approx.f32 %0, %1;" : "=f"(y) : "f"(x));
    return y;
}

template <bool FTZ>
__device__ __forceinline__ float sqrt_approx(float x) {
    float y;
    if (FTZ)
        asm("sqrt.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
    else
        asm("sqrt.approx.f32 %0, %1;" : "=f"(y) : "f"(x));
    return y;
}

// Smallest eps for which the flush-to-zero forms are exact substitutes.
constexpr float kFtzSafeEps = 1.17549435e-38f;  // 2^-126

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
// STD selects the prose reading of Sec. 2.2: v averages the std itself
// (r = sqrt(max(n - b^2, 0) + eps)) and the step divides by it.  With
// eps >= 2^-126 the std is >= 2^-63 and v >= 2^-87, so the flush-to-zero
// forms stay exact substitutes there too.
template <bool FTZ = false, bool STD = false>
__device__ __forceinline__ void fasgd_update(float& theta, float& n, float& b, float& v,
                                             float g, float coef, const StatParams& sp) {
    n = __fadd_rn(__fmul_rn(sp.gamma, n), __fmul_rn(sp.one_m_gamma, __fmul_rn(g, g)));
    b = __fadd_rn(__fmul_rn(sp.gamma, b), __fmul_rn(sp.one_m_gamma, g));
    const float var = fmaxf(__fsub_rn(n, __fmul_rn(b, b)), 0.0f);
    const float rad = __fadd_rn(var, sp.eps);
    const float r = STD ? sqrt_approx<FTZ>(rad) : rsqrt_approx<FTZ>(rad);
    v = fmaf(sp.beta, v, sp.one_m_beta * r);
    theta = fmaf(-(coef * g), rcp_approx<FTZ>(v), theta);
}

// The same rule with every operation correctly rounded and none fused
// (IEEE square root and division, separate multiplies and adds): the exact
// fp32 sequence Eq. 4-8 define, bit for bit on any IEEE machine.  Selected
// per handle (fasgd_set_exact) where results must be reproducible bit for
// bit, e.g. in closed-loop simulations; it costs a division and a square
// root per element-push on the pipes the fast form leaves idle.
template <bool STD = false>
__device__ __forceinline__ void fasgd_update_exact(float& theta, float& n, float& b, float& v,
                                                   float g, float coef, const StatParams& sp) {
    n = __fadd_rn(__fmul_rn(sp.gamma, n), __fmul_rn(sp.one_m_gamma, __fmul_rn(g, g)));
    b = __fadd_rn(__fmul_rn(sp.gamma, b), __fmul_rn(sp.one_m_gamma, g));
    const float var = fmaxf(__fsub_rn(n, __fmul_rn(b, b)), 0.0f);
    const float root = __fsqrt_rn(__fadd_rn(var, sp.eps));
    const float r = STD ? root : __fdiv_rn(1.0f, root);
    v = __fadd_rn(__fmul_rn(sp.beta, v), __fmul_rn(sp.one_m_beta, r));
    theta = __fsub_rn(theta, __fdiv_rn(__fmul_rn(coef, g), v));
}

// Arithmetic of a pass: hardware approximations (subnormal-preserving or
// flush-to-zero forms) or the exact sequence.
enum : int { kArithApprox = 0, kArithApproxFtz = 1, kArithExact = 2 };

template <int ARITH, bool STD>
__device__ __forceinline__ void rule_update(float& theta, float& n, float& b, float& v, float g,
                                            float coef, const StatParams& sp) {
    if (ARITH == kArithExact)
        fasgd_update_exact<STD>(theta, n, b, v, g, coef, sp);
    else
        fasgd_update<ARITH == kArithApproxFtz, STD>(theta, n, b, v, g, coef, sp);
}

}  // namespace fasgd
