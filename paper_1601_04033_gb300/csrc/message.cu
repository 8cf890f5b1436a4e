// The paper's literal B-FASGD (Sec. 2.3): one Eq. 9 decision per
// transmission opportunity, taken against v = the mean over all parameters
// of the server's moving averages.
//
// Two kernels per decision:
//   1. vbar_partial: the parameters are cut into 128-parameter chunks and
//      the chunks into one contiguous range per block; each block combines
//      its chunks' float-float sums in a fixed order into one partial.  The
//      chunk sums are those the dense pass leaves after a message push (so
//      v is not read again), or, when another pass has changed v since, the
//      block forms them from v with the same arithmetic and stores them;
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
// fetch, src is theta and dst the client's copy.  Under the FASGD rules a
// push skips kernel 2: the pass that applies it takes the same decision
// (message_decide, message.cuh) and refreshes the slot as it streams
// (dense.cu); kernel 2 serves fetches, the statistic query and ASGD/SASGD
// pushes.

#include "eq9.cuh"
#include "kernels.cuh"
#include "message.cuh"
#include "pdl.cuh"
#include "twosum.cuh"

namespace fasgd {
namespace {

constexpr int kMsgThreads = 256;

// This lane's four values of chunk c of v (parameters 4 lane .. 4 lane + 3
// of the chunk), zeros past P.  chunk_sum4 over them gives the same bits the
// dense pass leaves for the chunk.
__device__ __forceinline__ float4 chunk_values(const float* v, int64_t P, int64_t c, int lane) {
    const int64_t e = c * kVsumChunk + 4 * lane;
    if (e + 3 < P) return __ldcs(reinterpret_cast<const float4*>(v + e));
    float4 x;
    x.x = e < P ? v[e] : 0.f;
    x.y = e + 1 < P ? v[e + 1] : 0.f;
    x.z = e + 2 < P ? v[e + 2] : 0.f;
    x.w = e + 3 < P ? v[e + 3] : 0.f;
    return x;
}

// Block b combines chunks [c0, c1) in a fixed order: chunk c0 + w + 8 i goes
// to warp w, slot i, and lane (i mod 32) of that warp adds its slots in
// increasing i; then each warp's tree, then the warps in order.  from_v: the
// warp forms each chunk sum from v (four chunks' loads in flight) and stores
// it; otherwise lane l loads its slots' stored sums.  Both give the same bits.
__global__ void __launch_bounds__(kMsgThreads) vbar_partial_kernel(const __grid_constant__ MessageArgs a) {
    __shared__ float2 smem[kMsgThreads / 32];
    pdl_wait();
    pdl_trigger();
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    constexpr int kWarps = kMsgThreads / 32;
    const int64_t nch = (a.P + kVsumChunk - 1) / kVsumChunk;
    const int64_t per = (nch + a.nblocks - 1) / a.nblocks;
    const int64_t c0 = (int64_t)blockIdx.x * per;
    const int64_t c1 = c0 + per < nch ? c0 + per : nch;
    const int64_t nslots = c1 > c0 + warp ? (c1 - c0 - warp + kWarps - 1) / kWarps : 0;
    float h = 0.f, l = 0.f;
    if (a.from_v) {
        for (int64_t i0 = 0; i0 < nslots; i0 += 4) {
            float4 x[4];
#pragma unroll
            for (int k = 0; k < 4; ++k)
                if (i0 + k < nslots) x[k] = chunk_values(a.v, a.P, c0 + warp + kWarps * (i0 + k), lane);
#pragma unroll
            for (int k = 0; k < 4; ++k) {
                const int64_t i = i0 + k;
                if (i < nslots) {   // warp-uniform: the tree below uses every lane
                    const int64_t c = c0 + warp + kWarps * i;
                    const float2 cs = chunk_sum4(x[k]);
                    if (lane == 0) a.chunks[c] = cs;
                    if (lane == (int)(i & 31)) ff_add(h, l, cs.x, cs.y);
                }
            }
        }
    } else {
        for (int64_t i0 = lane; i0 < nslots; i0 += 4 * 32) {
            float2 x[4];
#pragma unroll
            for (int k = 0; k < 4; ++k)
                if (i0 + 32 * k < nslots) x[k] = a.chunks[c0 + warp + kWarps * (i0 + 32 * k)];
#pragma unroll
            for (int k = 0; k < 4; ++k)
                if (i0 + 32 * k < nslots) ff_add(h, l, x[k].x, x[k].y);
        }
    }
    ff_warp_sum(h, l);
    if (lane == 0) smem[warp] = make_float2(h, l);
    __syncthreads();
    if (threadIdx.x == 0) {
        float2 t = make_float2(0.f, 0.f);
        for (int w = 0; w < kWarps; ++w) ff_add(t.x, t.y, smem[w].x, smem[w].y);
        a.partial[blockIdx.x] = t;
    }
}

__global__ void __launch_bounds__(kMsgThreads) message_resolve_kernel(const __grid_constant__ MessageArgs a) {
    __shared__ uint32_t s_send;
    pdl_wait();
    pdl_trigger();
    if (threadIdx.x < 32) {
        float vbar;
        const uint32_t send = message_decide(a.partial, a.nblocks, a.P, a.c, a.eps_b,
                                             a.round_key0, a.round_key1, a.client_word, a.n_lo,
                                             a.n_hi, &vbar);
        if (threadIdx.x == 0) {
            s_send = send;
            if (blockIdx.x == 0 && a.flag_out != nullptr) *a.flag_out = (int32_t)send;
            if (blockIdx.x == 0 && a.vbar_out != nullptr) *a.vbar_out = vbar;
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
    const int64_t nch = (P + kVsumChunk - 1) / kVsumChunk;
    int64_t b = (nch + 255) / 256;   // ~256 chunks (32,768 parameters) per block
    if (b < 1) b = 1;
    if (b > kMessageMaxBlocks) b = kMessageMaxBlocks;
    return (int32_t)b;
}

cudaError_t launch_message_partials(const MessageArgs& a, cudaStream_t stream, int64_t* launches) {
    const cudaError_t st = launch_pdl(vbar_partial_kernel, a.nblocks, kMsgThreads, 0, stream, a);
    if (st == cudaSuccess) ++*launches;
    return st;
}

cudaError_t launch_message(const MessageArgs& a, int num_sms, cudaStream_t stream,
                           int64_t* launches) {
    cudaError_t st = launch_message_partials(a, stream, launches);
    if (st != cudaSuccess) return st;
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
