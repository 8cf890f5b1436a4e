// Sparse server apply of one B-FASGD push (paper Sec. 2.3 with unsent
// entries dropped): for i < count, parameter p = idx[i] receives gradient
// entry val[i] through the same per-element rule as the dense pass
// (Eq. 1-2 or Eq. 4-8); parameters not in the list are not touched.
//
// Indices in one list are strictly ascending, so no two threads touch the
// same parameter and no atomics are needed.  The count is read on the device
// (it was produced there by the select kernels), so no host round trip sits
// between select and apply.  A persistent grid walks the list; each warp
// takes 32 consecutive entries per step, four steps per iteration, so the
// index and value loads are coalesced and four gathers per array are in
// flight per thread.

#include <atomic>

#include "kernels.cuh"
#include "pdl.cuh"
#include "update.cuh"

namespace fasgd {
namespace {

constexpr int kSparseThreads = 256;
constexpr int kUnroll = 4;

template <int RULE, bool EXACT>
__global__ void __launch_bounds__(kSparseThreads) fasgd_sparse_kernel(const __grid_constant__ SparseArgs a) {
    constexpr bool FAS = RULE != kRuleSgd;
    pdl_wait();
    pdl_trigger();
    int64_t count = a.count_max;
    if (a.count_dev != nullptr) {
        const int64_t c = *a.count_dev;
        count = c;
        if (c < 0 || c > a.count_max) {
            if (blockIdx.x == 0 && threadIdx.x == 0) atomicOr(a.err, 1);
            count = c < 0 ? 0 : a.count_max;
        }
    }
    const int lane = threadIdx.x & 31;
    const int64_t warp_id = ((int64_t)blockIdx.x * kSparseThreads + threadIdx.x) >> 5;
    const int64_t nwarps = ((int64_t)gridDim.x * kSparseThreads) >> 5;
    for (int64_t base = warp_id * (32 * kUnroll); base < count; base += nwarps * (32 * kUnroll)) {
        int32_t p[kUnroll];
        float g[kUnroll];
        bool ok[kUnroll];
#pragma unroll
        for (int u = 0; u < kUnroll; ++u) {
            const int64_t i = base + u * 32 + lane;
            ok[u] = false;
            p[u] = 0;
            g[u] = 0.f;
            if (i < count) {
                p[u] = a.idx[i];
                g[u] = a.val[i];
                const int32_t prev = (i > 0) ? a.idx[i - 1] : -1;
                if (p[u] < 0 || (int64_t)p[u] >= a.P) {
                    atomicOr(a.err, 2);
                } else if (p[u] <= prev) {
                    atomicOr(a.err, 4);
                } else {
                    ok[u] = true;
                }
            }
        }
        float th[kUnroll], n[kUnroll], b[kUnroll], v[kUnroll];
#pragma unroll
        for (int u = 0; u < kUnroll; ++u) {
            if (ok[u]) {
                th[u] = a.theta[p[u]];
                if (FAS) {
                    n[u] = a.n[p[u]];
                    b[u] = a.b[p[u]];
                    v[u] = a.v[p[u]];
                }
            }
        }
#pragma unroll
        for (int u = 0; u < kUnroll; ++u) {
            if (ok[u]) {
                if (FAS) {
                    rule_update<EXACT ? kArithExact : kArithApprox, RULE == kRuleFasgdStd>(
                        th[u], n[u], b[u], v[u], g[u], a.coef, a.sp);
                    a.n[p[u]] = n[u];
                    a.b[p[u]] = b[u];
                    a.v[p[u]] = v[u];
                } else {
                    sgd_update(th[u], g[u], a.coef);
                }
                a.theta[p[u]] = th[u];
            }
        }
    }
}

template <int RULE, bool EXACT>
cudaError_t launch_rule(const SparseArgs& a, int num_sms, cudaStream_t stream) {
    // Resident blocks per SM, looked up once (the grid is only capped by it).
    static std::atomic<int> cached{0};
    int blocks_per_sm = cached.load(std::memory_order_relaxed);
    if (blocks_per_sm == 0) {
        cudaError_t st = cudaOccupancyMaxActiveBlocksPerMultiprocessor(
            &blocks_per_sm, fasgd_sparse_kernel<RULE, EXACT>, kSparseThreads, 0);
        if (st != cudaSuccess) return st;
        if (blocks_per_sm < 1) blocks_per_sm = 1;
        cached.store(blocks_per_sm, std::memory_order_relaxed);
    }
    // Enough warps for the host-side bound on the count, at most one full wave.
    const int64_t per_block = (int64_t)kSparseThreads * kUnroll;
    int64_t want = (a.count_max + per_block - 1) / per_block;
    const int64_t cap = (int64_t)num_sms * blocks_per_sm;
    if (want > cap) want = cap;
    if (want < 1) want = 1;
    return launch_pdl(fasgd_sparse_kernel<RULE, EXACT>, (unsigned)want, kSparseThreads, 0, stream, a);
}

constexpr int kScatterUnroll = 8;

// Client side of a B-FASGD fetch: theta[idx[i]] = val[i] for i < count.
// Indices come from one compaction, so they are distinct and no two threads
// write the same parameter; an index outside [0, P) is skipped and flagged.
__global__ void __launch_bounds__(kSparseThreads) fetch_scatter_kernel(const __grid_constant__ ScatterArgs a) {
    pdl_wait();
    pdl_trigger();
    int64_t count = a.count_max;
    if (a.count_dev != nullptr) {
        const int64_t c = *a.count_dev;
        count = c;
        if (c < 0 || c > a.count_max) {
            if (blockIdx.x == 0 && threadIdx.x == 0 && a.err != nullptr) atomicOr(a.err, 1);
            count = c < 0 ? 0 : a.count_max;
        }
    }
    // kScatterUnroll entries per thread per step (consecutive lanes, coalesced
    // list loads), every load of a step issued before its stores.
    const int64_t span = (int64_t)kSparseThreads * kScatterUnroll;
    for (int64_t base = (int64_t)blockIdx.x * span; base < count; base += (int64_t)gridDim.x * span) {
        int32_t p[kScatterUnroll];
        float x[kScatterUnroll];
#pragma unroll
        for (int k = 0; k < kScatterUnroll; ++k) {
            const int64_t i = base + k * kSparseThreads + threadIdx.x;
            p[k] = 0;
            x[k] = 0.f;
            if (i < count) {
                p[k] = a.idx[i];
                x[k] = a.val[i];
            }
        }
#pragma unroll
        for (int k = 0; k < kScatterUnroll; ++k) {
            const int64_t i = base + k * kSparseThreads + threadIdx.x;
            if (i >= count) continue;
            if (p[k] < 0 || (int64_t)p[k] >= a.P) {
                if (a.err != nullptr) atomicOr(a.err, 2);
                continue;
            }
            a.theta[p[k]] = x[k];
        }
    }
}

}  // namespace

cudaError_t launch_scatter(const ScatterArgs& a, int num_sms, cudaStream_t stream) {
    const int64_t per_block = (int64_t)kSparseThreads * kScatterUnroll;
    int64_t want = (a.count_max + per_block - 1) / per_block;
    const int64_t cap = (int64_t)(num_sms > 0 ? num_sms : 1) * 8;
    if (want > cap) want = cap;
    if (want < 1) want = 1;
    return launch_pdl(fetch_scatter_kernel, (unsigned)want, kSparseThreads, 0, stream, a);
}

cudaError_t launch_sparse(const SparseArgs& a, int rule, bool exact, int num_sms,
                          cudaStream_t stream, int64_t* launches) {
    cudaError_t st;
    if (rule == kRuleSgd)
        st = launch_rule<kRuleSgd, false>(a, num_sms, stream);
    else if (rule == kRuleFasgd)
        st = exact ? launch_rule<kRuleFasgd, true>(a, num_sms, stream)
                   : launch_rule<kRuleFasgd, false>(a, num_sms, stream);
    else
        st = exact ? launch_rule<kRuleFasgdStd, true>(a, num_sms, stream)
                   : launch_rule<kRuleFasgdStd, false>(a, num_sms, stream);
    if (st == cudaSuccess) ++*launches;
    return st;
}

}  // namespace fasgd
