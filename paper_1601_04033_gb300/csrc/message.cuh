// Internal interface of the per-message B-FASGD kernels (message.cu) for the
// host runtime.  Not part of the public C ABI.
#pragma once
#include "kernels.cuh"

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

}  // namespace fasgd
