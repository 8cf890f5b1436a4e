// Fused dense server pass: K pending pushes applied in one sweep over P.
//
// Each thread owns four consecutive parameters at a time (128-bit loads and
// stores).  theta (and n, b, v for FASGD) are loaded once, the K gradient
// slices are streamed in groups of G, every push is applied in arrival order
// with the state held in registers, and the state is stored once.  The pass
// therefore moves (8 + 4K) bytes per parameter for ASGD/SASGD and
// (32 + 4K) for FASGD, the minimum for K pushes (paper Sec. 2.1 protocol,
// Eq. 1-2 and Eq. 4-8 applied K times).
//
// Elements are independent, so the result does not depend on the grid: the
// per-element operation sequence is the same for every launch shape.

#include "kernels.cuh"
#include "update.cuh"

namespace fasgd {
namespace {

constexpr int kDenseThreads = 256;

__device__ __forceinline__ float4 ld_state(const float* p) {
    return *reinterpret_cast<const float4*>(p);
}

__device__ __forceinline__ void st_state(float* p, const float4& x) {
    *reinterpret_cast<float4*>(p) = x;
}

// Gradient slices are read exactly once: streaming (evict-first) loads.
__device__ __forceinline__ float4 ld_grad(const float* p) {
    return __ldcs(reinterpret_cast<const float4*>(p));
}

template <bool FAS>
__device__ __forceinline__ void update4(float4& th, float4& n, float4& b, float4& v,
                                        const float4& g, float coef, const StatParams& sp) {
    if (FAS) {
        fasgd_update(th.x, n.x, b.x, v.x, g.x, coef, sp);
        fasgd_update(th.y, n.y, b.y, v.y, g.y, coef, sp);
        fasgd_update(th.z, n.z, b.z, v.z, g.z, coef, sp);
        fasgd_update(th.w, n.w, b.w, v.w, g.w, coef, sp);
    } else {
        sgd_update(th.x, g.x, coef);
        sgd_update(th.y, g.y, coef);
        sgd_update(th.z, g.z, coef);
        sgd_update(th.w, g.w, coef);
    }
}

template <bool FAS, int G>
__global__ void __launch_bounds__(kDenseThreads)
fasgd_dense_kernel(const __grid_constant__ DenseArgs a) {
    const int64_t nquads = a.P >> 2;
    const int64_t stride = (int64_t)gridDim.x * kDenseThreads;
    const int K = a.K;
    for (int64_t q = (int64_t)blockIdx.x * kDenseThreads + threadIdx.x; q < nquads; q += stride) {
        const int64_t e = q << 2;
        float4 th = ld_state(a.theta + e);
        float4 n = make_float4(0.f, 0.f, 0.f, 0.f), b = n, v = n;
        if (FAS) {
            n = ld_state(a.n + e);
            b = ld_state(a.b + e);
            v = ld_state(a.v + e);
        }
        int k0 = 0;
        for (; k0 + G <= K; k0 += G) {
            float4 g[G];
#pragma unroll
            for (int j = 0; j < G; ++j) g[j] = ld_grad(a.grad[k0 + j] + e);
#pragma unroll
            for (int j = 0; j < G; ++j) update4<FAS>(th, n, b, v, g[j], a.coef[k0 + j], a.sp);
        }
        if (k0 < K) {  // last, partial group
            float4 g[G];
#pragma unroll
            for (int j = 0; j < G; ++j)
                if (k0 + j < K) g[j] = ld_grad(a.grad[k0 + j] + e);
#pragma unroll
            for (int j = 0; j < G; ++j)
                if (k0 + j < K) update4<FAS>(th, n, b, v, g[j], a.coef[k0 + j], a.sp);
        }
        st_state(a.theta + e, th);
        if (FAS) {
            st_state(a.n + e, n);
            st_state(a.b + e, b);
            st_state(a.v + e, v);
        }
    }
    // Ragged tail: the last P mod 4 parameters, one per thread of the last block.
    const int rem = (int)(a.P & 3);
    if (rem != 0 && blockIdx.x == gridDim.x - 1 && (int)threadIdx.x < rem) {
        const int64_t p = (nquads << 2) + threadIdx.x;
        float th = a.theta[p];
        float n = 0.f, b = 0.f, v = 0.f;
        if (FAS) {
            n = a.n[p];
            b = a.b[p];
            v = a.v[p];
        }
        for (int k = 0; k < K; ++k) {
            const float g = __ldcs(a.grad[k] + p);
            if (FAS)
                fasgd_update(th, n, b, v, g, a.coef[k], a.sp);
            else
                sgd_update(th, g, a.coef[k]);
        }
        a.theta[p] = th;
        if (FAS) {
            a.n[p] = n;
            a.b[p] = b;
            a.v[p] = v;
        }
    }
}

template <bool FAS, int G>
cudaError_t launch_g(const DenseArgs& a, int num_sms, cudaStream_t stream) {
    static int blocks_per_sm = 0;  // resident blocks of this instantiation, queried once
    if (blocks_per_sm == 0) {
        cudaError_t st = cudaOccupancyMaxActiveBlocksPerMultiprocessor(
            &blocks_per_sm, fasgd_dense_kernel<FAS, G>, kDenseThreads, 0);
        if (st != cudaSuccess) return st;
        if (blocks_per_sm < 1) blocks_per_sm = 1;
    }
    const int64_t nquads = a.P >> 2;
    int64_t want = (nquads + kDenseThreads - 1) / kDenseThreads;
    const int64_t cap = (int64_t)num_sms * blocks_per_sm;
    if (want > cap) want = cap;
    if (want < 1) want = 1;
    fasgd_dense_kernel<FAS, G><<<(unsigned)want, kDenseThreads, 0, stream>>>(a);
    return cudaGetLastError();
}

template <bool FAS>
cudaError_t launch_rule(const DenseArgs& a, int num_sms, cudaStream_t stream) {
    // Group size: the largest power of two <= K, at most 16.
    if (a.K >= 16) return launch_g<FAS, 16>(a, num_sms, stream);
    if (a.K >= 8) return launch_g<FAS, 8>(a, num_sms, stream);
    if (a.K >= 4) return launch_g<FAS, 4>(a, num_sms, stream);
    if (a.K >= 2) return launch_g<FAS, 2>(a, num_sms, stream);
    return launch_g<FAS, 1>(a, num_sms, stream);
}

}  // namespace

cudaError_t launch_dense(const DenseArgs& a, bool fasgd_rule, int num_sms, cudaStream_t stream,
                         int64_t* launches) {
    cudaError_t st = fasgd_rule ? launch_rule<true>(a, num_sms, stream)
                                : launch_rule<false>(a, num_sms, stream);
    if (st == cudaSuccess) ++*launches;
    return st;
}

}  // namespace fasgd
