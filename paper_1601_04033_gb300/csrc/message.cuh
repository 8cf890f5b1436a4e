// Internal interface of the per-message B-FASGD kernels (message.cu) for the
// host runtime.  Not part of the public C ABI.
#pragma once
#include "eq9.cuh"
#include "kernels.cuh"
#include "twosum.cuh"

namespace fasgd {

// One per-message B-FASGD decision (push or fetch) and, when the message is
// transmitted, the copy src -> dst (P floats, both 16-byte aligned).
constexpr int kMessageMaxBlocks = 1024;

struct MessageArgs {
    const float* v;            // the server's statistic, fp32[P]
    int64_t P;
    float2* partial;           // scratch: nblocks float-float partial sums
    int32_t nblocks;           // message_partial_blocks(P)
    float2* chunks;            // ceil(P / 128) chunk sums of v
    int32_t from_v;            // 1: form the chunk sums from v (and store them);
                               // 0: they are current (left by the dense pass)
    float c;                   // c_push or c_fetch
    float eps_b;
    uint32_t round_key0[10];
    uint32_t round_key1[10];
    uint32_t client_word;      // client + 2^31 * stream (0: push, 1: fetch)
    uint32_t n_lo, n_hi;       // the client's count of earlier messages of that stream
    const float* src;          // may be null: decide only
    float* dst;
    int32_t* flag_out;         // may be null: 1 transmitted, 0 dropped
    float* vbar_out;           // may be null: the statistic vbar the decision used
};

int32_t message_partial_blocks(int64_t P);

cudaError_t launch_message(const MessageArgs& a, int num_sms, cudaStream_t stream,
                           int64_t* launches);
// The partials only (vbar_partial_kernel): for a decision the pass that
// follows takes itself (message_decide).
cudaError_t launch_message_partials(const MessageArgs& a, cudaStream_t stream, int64_t* launches);

// The decision of one message from the nblocks partials vbar_partial_kernel
// left, taken by one whole warp: lane l adds partials l, l + 32, ... in
// order (eight loads in flight), then a fixed float-float shuffle tree,
// vbar = fl32(sum / P) (ff_div_int), u = word 0 of Philox4x32-10 at counter
// (2^32-1, client_word, n_lo, n_hi), the exact Eq. 9 test.  Every caller
// forms the same bits.  Returns the decision (1: transmitted) in every lane
// and vbar in *vbar.
__device__ __forceinline__ uint32_t message_decide(const float2* partial, int32_t nblocks,
                                                   int64_t P, float c, float eps_b,
                                                   const uint32_t (&rk0)[10],
                                                   const uint32_t (&rk1)[10],
                                                   uint32_t client_word, uint32_t n_lo,
                                                   uint32_t n_hi, float* vbar) {
    const int lane = threadIdx.x & 31;
    float h = 0.f, l = 0.f;
    for (int b = lane; b < nblocks; b += 8 * 32) {
        float2 x[8];
#pragma unroll
        for (int k = 0; k < 8; ++k)
            if (b + 32 * k < nblocks) x[k] = partial[b + 32 * k];
#pragma unroll
        for (int k = 0; k < 8; ++k)
            if (b + 32 * k < nblocks) ff_add(h, l, x[k].x, x[k].y);
    }
    ff_warp_sum(h, l);
    const float vb = ff_div_int(h, l, (int32_t)P);
    const Philox4 r = philox4x32_10(0xFFFFFFFFu, client_word, n_lo, n_hi, rk0, rk1);
    *vbar = vb;
    return send_bit(r.x[0] >> 8, vb, c, eps_b);
}

}  // namespace fasgd
