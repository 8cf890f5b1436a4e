// Compensated fp32 summation shared by the mean-of-v reductions.
#pragma once

#include <stdint.h>

namespace fasgd {

// hi + lo += x, with the rounding error of the fp32 addition recovered
// exactly (TwoSum: six operations, no branch, no contraction).  lo collects
// the errors in fp32 and is itself rounded, which bounds the pair's error by
// a few ulp of lo -- far below one ulp of the fp64 total.
__device__ __forceinline__ void two_sum_acc(float& hi, float& lo, float x) {
    const float t = __fadd_rn(hi, x);
    const float xp = __fsub_rn(t, hi);
    const float hp = __fsub_rn(t, xp);
    const float err = __fadd_rn(__fsub_rn(hi, hp), __fsub_rn(x, xp));
    lo = __fadd_rn(lo, err);
    hi = t;
}

// s + e = a + b exactly (Knuth's TwoSum).
__device__ __forceinline__ void two_sum(float a, float b, float& s, float& e) {
    s = __fadd_rn(a, b);
    const float bp = __fsub_rn(s, a);
    const float ap = __fsub_rn(s, bp);
    e = __fadd_rn(__fsub_rn(a, ap), __fsub_rn(b, bp));
}

// (h, l) += (h2, l2) for float-float pairs of non-negative sums: the sum of
// the high parts exactly, the low parts and that error added in fp32, then
// renormalised so that |l| <= ulp(h) / 2.  Relative error a few 2^-48 per
// addition for non-negative terms (no cancellation); pure fp32, so it runs
// on the full-width pipes (the fp64 pipe is narrow on this part).
__device__ __forceinline__ void ff_add(float& h, float& l, float h2, float l2) {
    float s, e;
    two_sum(h, h2, s, e);
    e = __fadd_rn(e, __fadd_rn(l, l2));
    two_sum(s, e, h, l);
}

// Warp-wide float-float sum over a fixed xor tree: every lane ends with the
// same pair.
__device__ __forceinline__ void ff_warp_sum(float& h, float& l) {
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) {
        const float h2 = __shfl_xor_sync(0xffffffffu, h, off);
        const float l2 = __shfl_xor_sync(0xffffffffu, l, off);
        ff_add(h, l, h2, l2);
    }
}

// The sum of one 128-parameter chunk of v, as a float-float pair, from this
// lane's four consecutive values (lane l holds parameters 4l .. 4l + 3 of the
// chunk; values past the end are passed as 0, which adds nothing): TwoSum in
// the order x, y, z, w, renormalised, then the fixed warp tree.  Every lane
// ends with the same pair; the bits depend only on the values.
__device__ __forceinline__ float2 chunk_sum4(float4 v) {
    float hi = 0.f, lo = 0.f;
    two_sum_acc(hi, lo, v.x);
    two_sum_acc(hi, lo, v.y);
    two_sum_acc(hi, lo, v.z);
    two_sum_acc(hi, lo, v.w);
    float h, l;
    two_sum(hi, lo, h, l);
    ff_warp_sum(h, l);
    return make_float2(h, l);
}

// fl32((h + l) / s) for a float-float pair (h >= 0, |l| <= ulp(h)) and an
// integer 1 <= s < 2^31, in fp32 only (the fp64 pipe is narrow here): with
// sh = fl(s) and sl = s - sh (exact, |sl| <= 64), q0 = fl(h / sh) leaves the
// residual h - q0 sh exactly representable (one fused multiply-add forms
// it); adding l and subtracting q0 sl rounds terms some 2^-20 of ulp(q0)
// small, so fl(q0 + r / sh) is the correctly rounded quotient except within
// about 2^-43 (relative) of a rounding boundary.
__device__ __forceinline__ float ff_div_int(float h, float l, int32_t s) {
    const float sh = __int2float_rn(s);
    // s - sh is an integer of magnitude at most 64 (sh may round up to 2^31,
    // so the difference is taken modulo 2^32 in unsigned arithmetic).
    const float sl = __int2float_rn((int32_t)((uint32_t)s - __float2uint_rn(sh)));
    const float q0 = __fdiv_rn(h, sh);
    const float e1 = __fmaf_rn(-q0, sh, h);
    const float r = __fsub_rn(__fadd_rn(e1, l), __fmul_rn(q0, sl));
    return __fadd_rn(q0, __fdiv_rn(r, sh));
}

}  // namespace fasgd
