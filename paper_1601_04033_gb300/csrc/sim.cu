// Closed-loop simulation support (the paper's FRED simulator, Sec. 3, with a
// synthetic objective standing in for its MNIST model): clients compute
// stochastic gradients of f(theta) = 1/2 sum_p h_p (theta_p - star_p)^2 on
// their own, possibly stale, copies of the parameters.
//
// Gradient: g_p = fl( fl(h_p (theta_p - star_p)) + fl(sigma_p xi_p) ) with
// uniform noise of unit variance xi_p = fl(x sqrt(12)), x = (u + 1/2) 2^-23 - 1/2
// exact, u = the top 23 bits of word (p mod 4) of Philox4x32-10 at counter
// (p div 4, client + 2^30, n, n >> 32) -- every operation exact or rounded
// once, so the result is reproducible bit for bit.
// Loss: the terms h (theta - star)^2 in fp32, summed over a fixed partition
// (per thread an fp32 sum plus its exact TwoSum errors, then fixed fp64
// combines), times 1/2.

#include "eq9.cuh"
#include "kernels.cuh"

namespace fasgd {
namespace {

constexpr int kSimThreads = 256;
constexpr int kLossBlocks = 1024;
constexpr unsigned kFull = 0xffffffffu;

__device__ __forceinline__ float sim_grad_one(float theta, float h, float star, float sigma,
                                              uint32_t word) {
    const float root12 = 3.46410161513775458705f;
    const uint32_t u = word >> 9;
    const float x = __fsub_rn(__fmul_rn(__fadd_rn((float)u, 0.5f), 1.0f / 8388608.0f), 0.5f);
    const float xi = __fmul_rn(x, root12);
    const float d = __fsub_rn(theta, star);
    return __fadd_rn(__fmul_rn(h, d), __fmul_rn(sigma, xi));
}

__global__ void __launch_bounds__(kSimThreads) sim_grad_kernel(const __grid_constant__ SimGradArgs a) {
    const int64_t nq = (a.P + 3) >> 2;
    const int64_t stride = (int64_t)gridDim.x * kSimThreads;
    for (int64_t q = (int64_t)blockIdx.x * kSimThreads + threadIdx.x; q < nq; q += stride) {
        const Philox4 r = philox4x32_10((uint32_t)q, a.client | (1u << 30), a.n_lo, a.n_hi,
                                        a.round_key0, a.round_key1);
        const int64_t e = q << 2;
        if (e + 3 < a.P) {
            const float4 th = *reinterpret_cast<const float4*>(a.theta + e);
            const float4 h = *reinterpret_cast<const float4*>(a.h + e);
            const float4 st = *reinterpret_cast<const float4*>(a.star + e);
            const float4 sg = *reinterpret_cast<const float4*>(a.sigma + e);
            float4 g;
            g.x = sim_grad_one(th.x, h.x, st.x, sg.x, r.x[0]);
            g.y = sim_grad_one(th.y, h.y, st.y, sg.y, r.x[1]);
            g.z = sim_grad_one(th.z, h.z, st.z, sg.z, r.x[2]);
            g.w = sim_grad_one(th.w, h.w, st.w, sg.w, r.x[3]);
            *reinterpret_cast<float4*>(a.grad + e) = g;
        } else {
            for (int j = 0; j < 4; ++j)
                if (e + j < a.P)
                    a.grad[e + j] = sim_grad_one(a.theta[e + j], a.h[e + j], a.star[e + j],
                                                 a.sigma[e + j], r.x[j]);
        }
    }
}

__device__ __forceinline__ void two_sum_acc(float& hi, float& lo, float x) {
    const float t = __fadd_rn(hi, x);
    const float xp = __fsub_rn(t, hi);
    const float hp = __fsub_rn(t, xp);
    lo = __fadd_rn(lo, __fadd_rn(__fsub_rn(hi, hp), __fsub_rn(x, xp)));
    hi = t;
}

__global__ void __launch_bounds__(kSimThreads) sim_loss_partial_kernel(const __grid_constant__ SimLossArgs a) {
    __shared__ double smem[kSimThreads / 32];
    const int64_t chunk = (a.P + kLossBlocks - 1) / kLossBlocks;
    const int64_t p0 = (int64_t)blockIdx.x * chunk;
    const int64_t p1 = p0 + chunk < a.P ? p0 + chunk : a.P;
    float hi = 0.f, lo = 0.f;
    for (int64_t p = p0 + threadIdx.x; p < p1; p += kSimThreads) {
        const float d = __fsub_rn(a.theta[p], a.star[p]);
        two_sum_acc(hi, lo, __fmul_rn(a.h[p], __fmul_rn(d, d)));
    }
    double s = (double)hi + (double)lo;
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) s += __shfl_xor_sync(kFull, s, off);
    if ((threadIdx.x & 31) == 0) smem[threadIdx.x >> 5] = s;
    __syncthreads();
    if (threadIdx.x == 0) {
        double t = 0.0;
        for (int w = 0; w < kSimThreads / 32; ++w) t += smem[w];
        a.partial[blockIdx.x] = t;
    }
}

__global__ void sim_loss_final_kernel(const __grid_constant__ SimLossArgs a) {
    const int lane = threadIdx.x;
    double s = 0.0;
    for (int b = lane; b < kLossBlocks; b += 32) s += a.partial[b];
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) s += __shfl_xor_sync(kFull, s, off);
    if (lane == 0) *a.loss = 0.5 * s;
}

}  // namespace

cudaError_t launch_sim_grad(const SimGradArgs& a, int num_sms, cudaStream_t stream) {
    int64_t grid = (((a.P + 3) >> 2) + kSimThreads - 1) / kSimThreads;
    const int64_t cap = (int64_t)(num_sms > 0 ? num_sms : 1) * 8;
    if (grid > cap) grid = cap;
    if (grid < 1) grid = 1;
    sim_grad_kernel<<<(unsigned)grid, kSimThreads, 0, stream>>>(a);
    return cudaGetLastError();
}

cudaError_t launch_sim_loss(const SimLossArgs& a, cudaStream_t stream) {
    sim_loss_partial_kernel<<<kLossBlocks, kSimThreads, 0, stream>>>(a);
    cudaError_t st = cudaGetLastError();
    if (st != cudaSuccess) return st;
    sim_loss_final_kernel<<<1, 32, 0, stream>>>(a);
    return cudaGetLastError();
}

}  // namespace fasgd
