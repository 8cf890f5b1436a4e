// Internal interface of the per-tensor B-FASGD kernels (tensors.cu) for the
// host runtime.  Not part of the public C ABI.
#pragma once
#include "kernels.cuh"

namespace fasgd {

// The partition is cut into work items: pieces of one tensor of at most
// tensor_chunk(P) parameters, in parameter order; the items of tensor t are
// item_begin[t] .. item_begin[t+1]-1.
struct TensorItem {
    int64_t start;    // first parameter
    int32_t len;      // parameters in the item (>= 1)
    int32_t tensor;   // tensor the item belongs to
};
inline int64_t tensor_chunk(int64_t P) {
    const int64_t c = (P + 8191) / 8192;   // at most ~8192 items besides one per tensor
    return c > 8192 ? c : 8192;
}
constexpr int kTensorResolveThreads = 1024;
// Dynamic shared memory of the decision kernel for n_items items and T tensors.
inline size_t tensor_resolve_smem(int32_t n_items, int32_t T) {
    return (size_t)n_items * 8 + (size_t)T * 8 + (size_t)T * 4 + (size_t)T * 4 +
           ((size_t)T + 1) * 4 + (size_t)T * 4 + (size_t)T;
}
struct TensorArgs {
    const float* v;               // the server's statistic, fp32[P]
    const TensorItem* items;
    int32_t n_items;
    const int32_t* item_begin;    // T + 1 entries
    const int32_t* sizes;         // T entries
    int32_t T;
    float2* partial;              // one float-float sum of v per item
    float eps_b;
    int64_t limit;                // min(budget, P) * 2^32
    uint32_t round_key0[10];
    uint32_t round_key1[10];
    uint32_t client_word;         // client + 2^31 * stream (0: push, 1: fetch)
    uint32_t n_lo, n_hi;          // the client's count of earlier calls of that stream
    uint8_t* sent;                // T decisions (handle-owned)
    float* c_out;                 // threshold (handle-owned)
    int64_t* count_out;           // parameters transmitted (handle-owned)
    uint8_t* user_sent;           // caller copies, each may be null
    float* user_c;
    int64_t* user_count;
    float* vbar_cache;            // T: vbar_t as last formed
    uint8_t* dirty;               // T: v of tensor t changed since vbar_t was formed
    long long* c_prev;            // bit pattern of this stream's last threshold (< 0: none)
    int32_t all_dirty;            // form every vbar_t afresh
    int32_t mark_dirty;           // the transmitted tensors' v is about to change (a push)
};
// The transmitted tensors of one decision: Eq. 4-8 (or Eq. 1-2) with grad,
// or (copy mode) dst <- src.
struct RangeArgs {
    float* theta;
    float* n;
    float* b;
    float* v;
    const float* grad;
    float coef;
    StatParams sp;
    const TensorItem* items;
    int32_t n_items;
    const uint8_t* sent;
    const float* src;
    float* dst;
    float2* partial;              // item sums to refresh after the update (may be null)
};
// sums_valid: the item sums in a.partial are those of the current v (else
// the partial kernel forms them first).
cudaError_t launch_tensor_decide(const TensorArgs& a, bool sums_valid, cudaStream_t stream,
                                 int64_t* launches);
cudaError_t launch_tensor_apply(const RangeArgs& a, int rule, bool exact, cudaStream_t stream,
                                int64_t* launches);
cudaError_t launch_tensor_copy(const RangeArgs& a, cudaStream_t stream, int64_t* launches);

}  // namespace fasgd
