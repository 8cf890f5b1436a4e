// The paper's literal B-FASGD (Sec. 2.3): one Eq. 9 decision per
// transmission opportunity, taken against v = the mean over all parameters
// of the server's moving averages.
//
// Two kernels per decision:
//   1. vbar_partial: fixed partition of the parameters into contiguous
//      chunks, one per block; each block sums its chunk of v (fixed order: per
//      thread in index order as an fp32 sum plus its exact rounding errors,
//      then a fixed float-float tree) into one float-float partial;
//   2. message_resolve: every block adds the partials in the same fixed order
//      (float-float), forms vbar = fl32(sum / P) (ff_div_int), draws u
//      (Philox4x32-10, word 0 at counter
//      (2^32-1, client + 2^31 * stream, n)), takes the exact Eq. 9 decision,
//      and, if the message is transmitted, copies src to dst (grid-stride,
//      128-bit); block 0 reports the decision.
// The partition depends on P only, so the decision is the same for every
// launch and every GPU.  For a push, src is the client's gradient and dst its
// slot of the server's gradient cache (the pass that follows reads the
// slot, so a dropped push re-applies the client's last sent gradient); for a
// fetch, src is theta and dst the client's copy.

#include "eq9.cuh"
#include "kernels.cuh"
#include "message.cuh"
#include "pdl.cuh"
#include "twosum.cuh"

namespace fasgd {
namespace {

constexpr int kMsgThreads = 256;

__global__ void __launch_bounds__(kMsgThreads) vbar_partial_kernel(const __grid_constant__ MessageArgs a) {
    __shared__ float2 smem[kMsgThreads / 32];
    pdl_wait();
    pdl_trigger();
    const int64_t nq = a.P >> 2;
    const int64_t chunk = (nq + a.nblocks - 1) / a.nblocks;
    const int64_t q0 = (int64_t)blockIdx.x * chunk;
    const int64_t q1 = q0 + chunk < nq ? q0 + chunk : nq;
    // Per thread: an fp32 sum with its exact rounding error carried alongside
    // (Knuth's TwoSum), four quads loaded before they are added.
    float hi = 0.f, lo = 0.f;
    const float4* v4 = reinterpret_cast<const float4*>(a.v);
    for (int64_t q = q0 + threadIdx.x; q < q1; q += 4 * kMsgThreads) {
        float4 x[4];
#pragma unroll
        for (int k = 0; k < 4; ++k)
            if (q + k * kMsgThreads < q1) x[k] = __ldcs(v4 + q + k * kMsgThreads);
#pragma unroll
        for (int k = 0; k < 4; ++k)
            if (q + k * kMsgThreads < q1) {
                two_sum_acc(hi, lo, x[k].x);
                two_sum_acc(hi, lo, x[k].y);
                two_sum_acc(hi, lo, x[k].z);
                two_sum_acc(hi, lo, x[k].w);
            }
    }
    if (blockIdx.x == 0 && threadIdx.x < (int)(a.P & 3)) two_sum_acc(hi, lo, a.v[4 * nq + threadIdx.x]);
    // Fixed float-float tree over the block (the fp64 pipe is narrow on this part).
    float h, l;
    two_sum(hi, lo, h, l);
    ff_warp_sum(h, l);
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    if (lane == 0) smem[warp] = make_float2(h, l);
    __syncthreads();
    if (threadIdx.x == 0) {
        float2 t = make_float2(0.f, 0.f);
        for (int w = 0; w < kMsgThreads / 32; ++w) ff_add(t.x, t.y, smem[w].x, smem[w].y);
        a.partial[blockIdx.x] = t;
    }
}

__global__ void __launch_bounds__(kMsgThreads) message_resolve_kernel(const __grid_constant__ MessageArgs a) {
    __shared__ uint32_t s_send;
    pdl_wait();
    pdl_trigger();
    if (threadIdx.x < 32) {
        const int lane = threadIdx.x;
        float h = 0.f, l = 0.f;
        // Lane l adds partials l, l + 32, ... in order, eight loads in flight.
        for (int b = lane; b < a.nblocks; b += 8 * 32) {
            float2 x[8];
#pragma unroll
            for (int k = 0; k < 8; ++k)
                if (b + 32 * k < a.nblocks) x[k] = a.partial[b + 32 * k];
#pragma unroll
            for (int k = 0; k < 8; ++k)
                if (b + 32 * k < a.nblocks) ff_add(h, l, x[k].x, x[k].y);
        }
        ff_warp_sum(h, l);
        if (lane == 0) {
            const float vbar = ff_div_int(h, l, (int32_t)a.P);
            const Philox4 r = philox4x32_10(0xFFFFFFFFu, a.client_word, a.n_lo, a.n_hi,
                                            a.round_key0, a.round_key1);
            const uint32_t send = send_bit(r.x[0] >> 8, vbar, a.c, a.eps_b);
            s_send = send;
            if (blockIdx.x == 0 && a.flag_out != nullptr) *a.flag_out = (int32_t)send;
        }
    }
    __syncthreads();
    if (!s_send || a.src == nullptr) return;
    const int64_t nq = a.P >> 2;
    const int64_t stride = (int64_t)gridDim.x * kMsgThreads;
    for (int64_t q = (int64_t)blockIdx.x * kMsgThreads + threadIdx.x; q < nq; q += stride)
        reinterpret_cast<float4*>(a.dst)[q] = __ldcs(reinterpret_cast<const float4*>(a.src) + q);
    if (blockIdx.x == 0 && threadIdx.x < (int)(a.P & 3))
        a.dst[4 * nq + threadIdx.x] = a.src[4 * nq + threadIdx.x];
}

}  // namespace

int32_t message_partial_blocks(int64_t P) {
    const int64_t nq = P >> 2;
    int64_t b = (nq + 8191) / 8192;  // ~8192 quads per block
    if (b < 1) b = 1;
    if (b > kMessageMaxBlocks) b = kMessageMaxBlocks;
    return (int32_t)b;
}

cudaError_t launch_message(const MessageArgs& a, int num_sms, cudaStream_t stream,
                           int64_t* launches) {
    cudaError_t st = launch_pdl(vbar_partial_kernel, a.nblocks, kMsgThreads, 0, stream, a);
    if (st != cudaSuccess) return st;
    ++*launches;
    int64_t grid = ((a.P >> 2) + kMsgThreads - 1) / kMsgThreads;
    const int64_t cap = (int64_t)(num_sms > 0 ? num_sms : 1) * 8;
    if (grid > cap) grid = cap;
    if (grid < 1) grid = 1;
    st = launch_pdl(message_resolve_kernel, (unsigned)grid, kMsgThreads, 0, stream, a);
    if (st != cudaSuccess) return st;
    ++*launches;
    return cudaSuccess;
}

}  // namespace fasgd
