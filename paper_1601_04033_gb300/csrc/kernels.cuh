// Internal interface between the host runtime (runtime.cu) and the kernels
// (dense.cu, select.cu, sparse.cu).  Not part of the public C ABI.
#pragma once

#include <cuda_runtime.h>
#include <stdint.h>

#include "fasgd.h"

namespace fasgd {

// Per-element update rule of a pass: ASGD/SASGD (Eq. 1-2), FASGD (Eq. 4-8),
// or FASGD with v averaging the std and the step divided by it (the prose
// reading of Sec. 2.2).
enum : int { kRuleSgd = 0, kRuleFasgd = 1, kRuleFasgdStd = 2 };

// Hyper-parameters of Eq. 4-6 as the kernels consume them.  one_m_gamma and
// one_m_beta are formed once on the host in fp32 (1 - gamma, 1 - beta).
struct StatParams {
    float gamma, one_m_gamma;
    float beta, one_m_beta;
    float eps;
};

// A per-message push decided inside its pass (with vsum, FASGD rules): the
// pass first takes the push's Eq. 9 decision from the statistic's partials
// (message_decide); if transmitted it applies src and copies it into slot
// (the client's gradient cache slot, which is also grad[0]), else it applies
// grad[0] as it stands.  partial == null: no decision, grad[0] is applied.
struct PassMessage {
    const float2* partial;          // nblocks float-float partial sums of v
    int32_t nblocks;
    float c, eps_b;
    uint32_t round_key0[10], round_key1[10];
    uint32_t client_word, n_lo, n_hi;
    const float* src;               // the pushed gradient, fp32[P], 16-byte aligned
    float* slot;                    // == grad[0]
    int32_t* flag_out;              // may be null: 1 transmitted, 0 dropped
};

// One fused pass over the parameters applying K dense pushes in order.
struct DenseArgs {
    float* theta;
    float* n;
    float* b;
    float* v;
    const float* grad[FASGD_KMAX];  // grad[k]: push k's gradient, fp32[P]
    float coef[FASGD_KMAX];         // alpha(tau_k) of push k (Eq. 1 / Eq. 7 without v)
    int64_t P;
    int32_t K;
    StatParams sp;
    int32_t* err;                   // device error flags (bit 3: a pipeline wait expired)
    float2* vsum;                   // if set (K = 1, FASGD rules): the float-float sum of
                                    // the new v over every 128-parameter chunk
    PassMessage msg;                // with vsum only
};
// Parameters per chunk of the per-message statistic's partial sums.
constexpr int kVsumChunk = 128;

// One sparse push: idx[i] receives val[i] for i < count.
struct SparseArgs {
    float* theta;
    float* n;
    float* b;
    float* v;
    const int32_t* idx;
    const float* val;
    const int64_t* count_dev;  // may be null: count = count_max
    int64_t count_max;
    int64_t P;
    float coef;
    StatParams sp;
    int32_t* err;              // device error flags (bit 0: count, bit 1: index, bit 2: order)
};

// Elements per tile of the select / compact kernels, and the bit mask words a
// tile owns (one bit per element).
constexpr int kSelectThreads = 256;
constexpr int kSelectTile = 8192;
constexpr int kSelectTileWords = kSelectTile / 32;

struct SelectArgs {
    const float* values;   // copied into val for kept parameters (a push's gradient, or theta)
    const float* v;
    int32_t* idx;
    float* val;
    int64_t* count;      // total number sent (int64, device)
    uint32_t* mask;      // scratch: ntiles * kSelectTileWords words
    int32_t* tile_count; // scratch: ntiles
    int64_t* tile_base;  // scratch: ntiles
    int64_t P;
    int32_t ntiles;
    float c;
    float eps_b;
    uint32_t round_key0[10];       // Philox key schedule: seed advanced by the
    uint32_t round_key1[10];       // Weyl constants, one pair per round
    uint32_t client_word;          // client + 2^31 * stream (0: push, 1: fetch)
    uint32_t push_lo, push_hi;     // the client's count of earlier calls of that stream
};

// Client side of a B-FASGD fetch: theta[idx[i]] = val[i] for i < count.
struct ScatterArgs {
    float* theta;
    const int32_t* idx;
    const float* val;
    const int64_t* count_dev;  // may be null: count = count_max
    int64_t count_max;
    int64_t P;
    int32_t* err;              // may be null; flags 1 (count) and 2 (index)
};

// Closed-loop simulation: stochastic gradient and loss of the synthetic
// quadratic objective (sim.cu).
struct SimGradArgs {
    const float* theta;   // the client's copy, fp32[P], 16-byte aligned
    const float* h;       // curvatures
    const float* star;    // minimiser
    const float* sigma;   // noise scales
    float* grad;          // output
    int64_t P;
    uint32_t round_key0[10];
    uint32_t round_key1[10];
    uint32_t client, n_lo, n_hi;
};

constexpr int kSimLossScratch = 1024;   // doubles of scratch the loss needs

struct SimLossArgs {
    const float* theta;
    const float* h;
    const float* star;
    int64_t P;
    double* partial;      // kSimLossScratch doubles
    double* loss;         // output (device)
};

// Launchers: enqueue on `stream`, return the launch status.
// `launches` is incremented by the number of kernels enqueued.
cudaError_t launch_dense(const DenseArgs& a, int rule, bool exact, int num_sms, cudaStream_t stream,
                         int64_t* launches);
cudaError_t launch_sparse(const SparseArgs& a, int rule, bool exact, int num_sms, cudaStream_t stream,
                          int64_t* launches);
cudaError_t launch_select(const SelectArgs& a, cudaStream_t stream, int64_t* launches);
cudaError_t launch_scatter(const ScatterArgs& a, int num_sms, cudaStream_t stream);
// Self-test: bounded pipeline waits that can never complete (raise flag 8 in err).
cudaError_t launch_wait_expiry(int32_t* err, cudaStream_t stream);
cudaError_t launch_sim_grad(const SimGradArgs& a, int num_sms, cudaStream_t stream);
cudaError_t launch_sim_loss(const SimLossArgs& a, cudaStream_t stream);

inline int32_t select_tiles(int64_t P) {
    return (int32_t)((P + kSelectTile - 1) / kSelectTile);
}

// Fills the Philox key schedule of `a` from the 64-bit seed.
void select_key_schedule(SelectArgs& a, uint64_t seed);

}  // namespace fasgd
