// Fused dense server pass: K pending pushes applied in one sweep over P.
//
// Every parameter's theta (and n, b, v for FASGD) is read once, the K
// gradient slices are read once, all K pushes are applied in arrival order
// with the state held in registers, and the state is written once.  The pass
// therefore moves (8 + 4K) bytes per parameter for ASGD/SASGD and (32 + 4K)
// for FASGD, the minimum for K pushes (paper Sec. 2.1 protocol, Eq. 1-2 and
// Eq. 4-8 applied K times).
//
// Structure: a persistent kernel, one block per SM, one producer warp and
// 16 consumer warps.  The parameter range is cut into tiles of 2048; the
// producer's elected lane stages each tile's state slices and up to 8
// gradient slices into a shared-memory ring with 1-D bulk async copies
// (cp.async.bulk, completion counted on an mbarrier), while the consumer
// warps compute on the previous stage: each thread takes four consecutive
// parameters (128-bit shared loads), frees the stage as soon as its inputs
// are in registers, applies the pushes, and stores the state with 128-bit
// global stores.  A stage holds up to 8 gradient slices; larger K runs as
// several stages per tile (the state travels with the first one only).  The
// last P mod 2048 parameters are handled by plain loads in the last block.
// Passes of fewer than 8 tiles per SM use a plain grid instead (one quad of
// parameters per thread, fasgd_direct_kernel).
//
// With SUMS (one push, a.vsum set) the pass also leaves the float-float sum
// of the new v over every 128-parameter chunk (one warp's share of a tile)
// in a.vsum, formed in registers, so the next per-message decision needs no
// pass over v (message.cu forms the same chunk sums from v, bit for bit).
// A SUMS pass of a per-message push also takes the push's Eq. 9 decision
// itself (a.msg: every block's warp 0 combines the statistic's partials in
// the decision kernel's order, message_decide) and, if the push is
// transmitted, applies the pushed gradient while copying it into the
// client's cache slot; if dropped it applies the slot.
//
// Both kernels are launched as programmatic dependents (pdl.cuh): a pass is
// scheduled while the kernel before it on the stream drains, sets up its
// barriers, and waits (griddepcontrol.wait) before it touches memory.
//
// Every wait on an mbarrier is bounded (about one second of wall clock);
// on expiry the block sets flag 8 of the error word, waits (bounded) for its
// own copies in flight, and returns.  Elements are independent, so the
// result does not depend on the grid or on which path handled an element.

#include <atomic>

#include "kernels.cuh"
#include "message.cuh"
#include "pdl.cuh"
#include "twosum.cuh"
#include "update.cuh"
#include "wait.cuh"

namespace fasgd {
namespace {

// Ring geometry per consumer count CONS (threads that compute; 512 or 256):
// tiles of 4 CONS parameters, CONS + 32 threads per block (one producer
// warp), 512 / CONS blocks per SM sharing 220 KB of shared memory.
template <int CONS> struct Geom {
    static constexpr int kTile = 4 * CONS;
    static constexpr int kThreads = CONS + 32;
    static constexpr int kBlocksPerSm = 512 / CONS;
    static constexpr int kSmemBudget = 220 * 1024 / kBlocksPerSm;   // ring + barriers, per block
};
constexpr int kTile = Geom<512>::kTile;         // the reference tile (2048 parameters)
constexpr int kMaxStages = 8;

// ---- bulk async copy (the mbarrier wrappers and bounded waits: wait.cuh) ----
// 1-D bulk copy global -> shared (16-byte aligned, size a multiple of 16),
// completion signalled on `bar` as transaction bytes.
__device__ __forceinline__ void bulk_load(void* dst, const void* src, uint32_t bytes, uint64_t* bar) {
    asm volatile(
        "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(
            smem_addr(dst)),
        "l"(src), "r"(bytes), "r"(smem_addr(bar))
        : "memory");
}

// ---- the element update on four consecutive parameters --------------------
template <int RULE, int ARITH>
__device__ __forceinline__ void update4(float4& th, float4& n, float4& b, float4& v, const float4& g,
                                        float coef, const StatParams& sp) {
    constexpr bool STD = RULE == kRuleFasgdStd;
    if (RULE != kRuleSgd) {
        rule_update<ARITH, STD>(th.x, n.x, b.x, v.x, g.x, coef, sp);
        rule_update<ARITH, STD>(th.y, n.y, b.y, v.y, g.y, coef, sp);
        rule_update<ARITH, STD>(th.z, n.z, b.z, v.z, g.z, coef, sp);
        rule_update<ARITH, STD>(th.w, n.w, b.w, v.w, g.w, coef, sp);
    } else {
        sgd_update(th.x, g.x, coef);
        sgd_update(th.y, g.y, coef);
        sgd_update(th.z, g.z, coef);
        sgd_update(th.w, g.w, coef);
    }
}

// Parameters [begin, P) with plain loads, by the CONS consumer threads of
// one block; begin is a multiple of 4.
template <int RULE, int ARITH, int CONS>
__device__ void apply_range_direct(const DenseArgs& a, int64_t begin, int tid) {
    constexpr bool FAS = RULE != kRuleSgd;
    const int64_t end_q = a.P & ~int64_t(3);
    for (int64_t e = begin + 4 * (int64_t)tid; e < end_q; e += 4 * (int64_t)CONS) {
        float4 th = *reinterpret_cast<const float4*>(a.theta + e);
        float4 n = make_float4(0.f, 0.f, 0.f, 0.f), b = n, v = n;
        if (FAS) {
            n = *reinterpret_cast<const float4*>(a.n + e);
            b = *reinterpret_cast<const float4*>(a.b + e);
            v = *reinterpret_cast<const float4*>(a.v + e);
        }
        for (int k = 0; k < a.K; ++k) {
            const float4 g = __ldcs(reinterpret_cast<const float4*>(a.grad[k] + e));
            update4<RULE, ARITH>(th, n, b, v, g, a.coef[k], a.sp);
        }
        *reinterpret_cast<float4*>(a.theta + e) = th;
        if (FAS) {
            *reinterpret_cast<float4*>(a.n + e) = n;
            *reinterpret_cast<float4*>(a.b + e) = b;
            *reinterpret_cast<float4*>(a.v + e) = v;
        }
    }
    const int64_t p = end_q + tid;  // the last P mod 4 parameters
    if (tid < (int)(a.P & 3) && p < a.P) {
        float th = a.theta[p], n = 0.f, b = 0.f, v = 0.f;
        if (FAS) {
            n = a.n[p];
            b = a.b[p];
            v = a.v[p];
        }
        for (int k = 0; k < a.K; ++k) {
            const float g = __ldcs(a.grad[k] + p);
            if (FAS)
                rule_update<ARITH, RULE == kRuleFasgdStd>(th, n, b, v, g, a.coef[k], a.sp);
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

// The SUMS form of the tail (one push): parameters [begin, P) chunk by
// chunk, consumer warp w taking chunks begin/128 + w, + CONS/32, ...; lane l
// updates parameters 4l .. 4l + 3 of the chunk (guarded at P) with gradient
// g0, copying it to copy_to unless that is null, and the warp forms the
// chunk's sum of the new v in registers.  begin is a multiple of 128.
template <int RULE, int ARITH, int CONS>
__device__ void apply_range_chunks(const DenseArgs& a, int64_t begin, int tid, const float* g0,
                                   float* copy_to) {
    const int warp = tid >> 5, lane = tid & 31;
    const int64_t nch = (a.P + kVsumChunk - 1) / kVsumChunk;
    for (int64_t c = begin / kVsumChunk + warp; c < nch; c += CONS / 32) {
        const int64_t e = c * kVsumChunk + 4 * lane;
        float th[4] = {0.f, 0.f, 0.f, 0.f}, n[4] = {0.f, 0.f, 0.f, 0.f};
        float b[4] = {0.f, 0.f, 0.f, 0.f}, v[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
        for (int j = 0; j < 4; ++j)
            if (e + j < a.P) {
                th[j] = a.theta[e + j];
                n[j] = a.n[e + j];
                b[j] = a.b[e + j];
                v[j] = a.v[e + j];
            }
#pragma unroll
        for (int j = 0; j < 4; ++j)
            if (e + j < a.P) {
                const float g = __ldcs(g0 + e + j);
                if (copy_to != nullptr) copy_to[e + j] = g;
                rule_update<ARITH, RULE == kRuleFasgdStd>(th[j], n[j], b[j], v[j], g, a.coef[0],
                                                          a.sp);
            }
#pragma unroll
        for (int j = 0; j < 4; ++j)
            if (e + j < a.P) {
                a.theta[e + j] = th[j];
                a.n[e + j] = n[j];
                a.b[e + j] = b[j];
                a.v[e + j] = v[j];
            }
        const float2 cs = chunk_sum4(make_float4(v[0], v[1], v[2], v[3]));
        if (lane == 0) a.vsum[c] = cs;
    }
}

// Ring geometry, identical on host and device.
struct Ring {
    int stages;     // stages in the ring
    int chunks;     // stages per tile: ceil(K / CH)
};

// RULE: kRuleSgd / kRuleFasgd / kRuleFasgdStd; ARITH: kArithApprox /
// kArithApproxFtz / kArithExact (see update.cuh); CH: gradient slices per stage;
// SUMS: also leave the chunk sums of the new v (FASGD rules, K = 1); CONS:
// consumer threads per block (the ring geometry, Geom).
template <int RULE, int ARITH, int CH, bool SUMS, int CONS>
__global__ void __launch_bounds__(Geom<CONS>::kThreads, Geom<CONS>::kBlocksPerSm)
fasgd_dense_kernel(const __grid_constant__ DenseArgs a, const Ring ring, const int64_t ntiles) {
    constexpr bool FAS = RULE != kRuleSgd;
    constexpr int kState = FAS ? 4 : 1;              // theta (, n, b, v)
    constexpr int kTile = Geom<CONS>::kTile;
    constexpr int kConsumers = CONS;
    constexpr int kStageFloats = (kState + CH) * kTile;
    extern __shared__ __align__(128) unsigned char smem[];
    float* buf = reinterpret_cast<float*>(smem);
    uint64_t* full = reinterpret_cast<uint64_t*>(smem + (size_t)ring.stages * kStageFloats * 4);
    uint64_t* empty = full + ring.stages;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    constexpr int kConsumerWarps = kConsumers / 32;

    if (threadIdx.x == 0) {
        for (int s = 0; s < ring.stages; ++s) {
            mbar_init(&full[s], 1);
            mbar_init(&empty[s], kConsumerWarps);
        }
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    }
    __syncthreads();
    pdl_wait();      // the kernel before this one on the stream is complete
    pdl_trigger();
    // A message push decided here (SUMS, a.msg.partial set): warp 0 takes the
    // decision, every thread reads it.  Transmitted: apply the pushed gradient
    // and copy it into the client's cache slot; dropped: apply the slot.
    const float* g0 = a.grad[0];
    float* copy_to = nullptr;
    if constexpr (SUMS) {
        __shared__ uint32_t s_send;
        if (a.msg.partial != nullptr) {
            if (warp == 0) {
                float vbar;
                const uint32_t send = message_decide(a.msg.partial, a.msg.nblocks, a.P, a.msg.c,
                                                     a.msg.eps_b, a.msg.round_key0,
                                                     a.msg.round_key1, a.msg.client_word,
                                                     a.msg.n_lo, a.msg.n_hi, &vbar);
                if (lane == 0) {
                    s_send = send;
                    if (blockIdx.x == 0 && a.msg.flag_out != nullptr) *a.msg.flag_out = (int32_t)send;
                }
            }
            __syncthreads();
            if (s_send) {
                g0 = a.msg.src;
                copy_to = a.msg.slot;
            }
        }
    }

    if (warp == kConsumerWarps) {
        // ---------------- producer: one elected lane ----------------
        if (lane == 0) {
            int s = 0;
            uint32_t ph = 0;
            bool ok = true;
            uint32_t issued = 0;            // bit s: stage s has been filled
            uint32_t issued_phase = 0;      // bit s: the phase parity of its last fill
            for (int64_t t = blockIdx.x; t < ntiles && ok; t += gridDim.x) {
                const int64_t off = t * kTile;
                for (int c = 0; c < ring.chunks; ++c) {
                    ok = wait_one(&empty[s], ph ^ 1u, a.err);
                    if (!ok) break;
                    const int k0 = c * CH;
                    const int ng = min(CH, a.K - k0);
                    const int ns = (c == 0) ? kState : 0;
                    mbar_arrive_expect_tx(&full[s], (uint32_t)((ns + ng) * kTile * 4));
                    float* st = buf + (size_t)s * kStageFloats;
                    if (ns > 0) {
                        bulk_load(st, a.theta + off, kTile * 4, &full[s]);
                        if (FAS) {
                            bulk_load(st + 1 * kTile, a.n + off, kTile * 4, &full[s]);
                            bulk_load(st + 2 * kTile, a.b + off, kTile * 4, &full[s]);
                            bulk_load(st + 3 * kTile, a.v + off, kTile * 4, &full[s]);
                        }
                    }
                    float* gs = st + kState * kTile;
                    for (int j = 0; j < ng; ++j)
                        bulk_load(gs + j * kTile, (k0 + j == 0 ? g0 : a.grad[k0 + j]) + off,
                                  kTile * 4, &full[s]);
                    issued |= 1u << s;
                    issued_phase = (issued_phase & ~(1u << s)) | (ph << s);
                    if (++s == ring.stages) {
                        s = 0;
                        ph ^= 1u;
                    }
                }
            }
            // Every fill issued by this block has landed before it exits.
            for (int i = 0; i < ring.stages; ++i)
                if (issued & (1u << i)) wait_one(&full[i], (issued_phase >> i) & 1u, a.err);
        }
        return;
    }

    // ---------------- consumers ----------------
    const int tid = threadIdx.x;
    int s = 0;
    uint32_t ph = 0;
    bool ok = true;
    for (int64_t t = blockIdx.x; t < ntiles && ok; t += gridDim.x) {
        float4 th = make_float4(0.f, 0.f, 0.f, 0.f), n = th, b = th, v = th;
        for (int c = 0; c < ring.chunks; ++c) {
            ok = wait_warp(&full[s], ph, a.err);
            if (!ok) break;
            const float* st = buf + (size_t)s * kStageFloats;
            if (c == 0) {
                th = reinterpret_cast<const float4*>(st)[tid];
                if (FAS) {
                    n = reinterpret_cast<const float4*>(st + 1 * kTile)[tid];
                    b = reinterpret_cast<const float4*>(st + 2 * kTile)[tid];
                    v = reinterpret_cast<const float4*>(st + 3 * kTile)[tid];
                }
            }
            const int k0 = c * CH;
            const float4* gs = reinterpret_cast<const float4*>(st + kState * kTile);
            float4 g[CH];
            if (k0 + CH <= a.K) {  // a full chunk
#pragma unroll
                for (int j = 0; j < CH; ++j) g[j] = gs[j * (kTile / 4) + tid];
                __syncwarp();
                if (lane == 0) mbar_arrive(&empty[s]);  // inputs are in registers
                if (SUMS && copy_to != nullptr)          // a transmitted message refreshes its slot
                    reinterpret_cast<float4*>(copy_to + t * kTile)[tid] = g[0];
#pragma unroll
                for (int j = 0; j < CH; ++j) update4<RULE, ARITH>(th, n, b, v, g[j], a.coef[k0 + j], a.sp);
            } else {               // the last, partial chunk
                const int ng = a.K - k0;
#pragma unroll
                for (int j = 0; j < CH; ++j)
                    if (j < ng) g[j] = gs[j * (kTile / 4) + tid];
                __syncwarp();
                if (lane == 0) mbar_arrive(&empty[s]);
#pragma unroll
                for (int j = 0; j < CH; ++j)
                    if (j < ng) update4<RULE, ARITH>(th, n, b, v, g[j], a.coef[k0 + j], a.sp);
            }
            if (++s == ring.stages) {
                s = 0;
                ph ^= 1u;
            }
        }
        if (!ok) break;
        const int64_t e = t * kTile + 4 * (int64_t)tid;
        *reinterpret_cast<float4*>(a.theta + e) = th;
        if (FAS) {
            *reinterpret_cast<float4*>(a.n + e) = n;
            *reinterpret_cast<float4*>(a.b + e) = b;
            *reinterpret_cast<float4*>(a.v + e) = v;
        }
        if (SUMS) {
            const float2 cs = chunk_sum4(v);
            if (lane == 0) a.vsum[(t * kTile) / kVsumChunk + warp] = cs;
        }
    }
    // Parameters after the last full tile.
    if (ok && blockIdx.x == gridDim.x - 1) {
        if (SUMS)
            apply_range_chunks<RULE, ARITH, CONS>(a, ntiles * kTile, tid, g0, copy_to);
        else
            apply_range_direct<RULE, ARITH, CONS>(a, ntiles * kTile, tid);
    }
}

template <int RULE, int ARITH, int CH, bool SUMS = false, int CONS = 512>
cudaError_t launch_ch(const DenseArgs& a, int num_sms, cudaStream_t stream) {
    using G = Geom<CONS>;
    constexpr int kState = RULE != kRuleSgd ? 4 : 1;
    constexpr int kStageBytes = (kState + CH) * G::kTile * 4;
    Ring ring;
    ring.chunks = (a.K + CH - 1) / CH;
    ring.stages = (G::kSmemBudget - 2 * kMaxStages * 8) / kStageBytes;
    if (ring.stages > kMaxStages) ring.stages = kMaxStages;
    const size_t smem = (size_t)ring.stages * kStageBytes + 2 * ring.stages * sizeof(uint64_t);
    // The shared-memory limit is a per-device attribute of the kernel: set it
    // once per device (bit d of the mask) and instantiation.
    static std::atomic<uint64_t> configured{0};
    int dev = 0;
    cudaError_t st = cudaGetDevice(&dev);
    if (st != cudaSuccess) return st;
    const uint64_t bit = dev < 64 ? 1ull << dev : 0;
    if (bit == 0 || !(configured.load(std::memory_order_acquire) & bit)) {
        st = cudaFuncSetAttribute(fasgd_dense_kernel<RULE, ARITH, CH, SUMS, CONS>,
                                  cudaFuncAttributeMaxDynamicSharedMemorySize, G::kSmemBudget);
        if (st != cudaSuccess) return st;
        configured.fetch_or(bit, std::memory_order_acq_rel);
    }
    const int64_t ntiles = a.P / G::kTile;
    // kBlocksPerSm blocks per SM (shared-memory bound), never more than there are tiles.
    const int64_t slots = (int64_t)G::kBlocksPerSm * num_sms;
    int64_t grid = ntiles < slots ? ntiles : slots;
    if (grid < 1) grid = 1;
    return launch_pdl(fasgd_dense_kernel<RULE, ARITH, CH, SUMS, CONS>, (unsigned)grid,
                      G::kThreads, smem, stream, a, ring, ntiles);
}

// ---- small passes ------------------------------------------------------------
// With few tiles per SM the ring's staging does not pay: its blocks stage,
// compute and store a handful of tiles each, and the last then runs the tail.
// A plain grid with one quad of parameters per thread and all of a thread's
// loads issued before its arithmetic makes one round trip to memory instead.
// Measured per pass (graph replay, K = 1 / 8): equal or faster up to
// 2.5M parameters (7,850: 2.1 / 3.4 us against 3.4 / 6.7 us; 1.29M: 5.0 /
// 10.7 us against 5.5 / 13.1 us), behind the ring from about 5M (K = 1:
// 23.5 against 18.1 us), so it takes passes below 8 tiles per SM.  Such
// working sets stay in L2 between passes, so the gradient loads keep the
// default cache policy here.
constexpr int kDirectThreads = 128;
constexpr int kDirectTilesPerSm = 8;

template <int RULE, int ARITH>
__global__ void __launch_bounds__(kDirectThreads)
fasgd_direct_kernel(const __grid_constant__ DenseArgs a) {
    constexpr bool FAS = RULE != kRuleSgd;
    constexpr bool STD = RULE == kRuleFasgdStd;
    pdl_wait();
    pdl_trigger();
    const int64_t nq = (a.P + 3) / 4;  // quads; the last may be partial
    for (int64_t q = (int64_t)blockIdx.x * kDirectThreads + threadIdx.x; q < nq;
         q += (int64_t)gridDim.x * kDirectThreads) {
        const int64_t e = 4 * q;
        if (e + 4 <= a.P) {
            float4 th = *reinterpret_cast<const float4*>(a.theta + e);
            float4 n = make_float4(0.f, 0.f, 0.f, 0.f), b = n, v = n;
            if (FAS) {
                n = *reinterpret_cast<const float4*>(a.n + e);
                b = *reinterpret_cast<const float4*>(a.b + e);
                v = *reinterpret_cast<const float4*>(a.v + e);
            }
            for (int k0 = 0; k0 < a.K; k0 += 8) {
                float4 g[8];
#pragma unroll
                for (int j = 0; j < 8; ++j)
                    if (k0 + j < a.K) g[j] = *reinterpret_cast<const float4*>(a.grad[k0 + j] + e);
#pragma unroll
                for (int j = 0; j < 8; ++j)
                    if (k0 + j < a.K) update4<RULE, ARITH>(th, n, b, v, g[j], a.coef[k0 + j], a.sp);
            }
            *reinterpret_cast<float4*>(a.theta + e) = th;
            if (FAS) {
                *reinterpret_cast<float4*>(a.n + e) = n;
                *reinterpret_cast<float4*>(a.b + e) = b;
                *reinterpret_cast<float4*>(a.v + e) = v;
            }
        } else {
            for (int64_t p = e; p < a.P; ++p) {
                float th = a.theta[p], n = 0.f, b = 0.f, v = 0.f;
                if (FAS) {
                    n = a.n[p];
                    b = a.b[p];
                    v = a.v[p];
                }
                for (int k = 0; k < a.K; ++k) {
                    if (FAS)
                        rule_update<ARITH, STD>(th, n, b, v, a.grad[k][p], a.coef[k], a.sp);
                    else
                        sgd_update(th, a.grad[k][p], a.coef[k]);
                }
                a.theta[p] = th;
                if (FAS) {
                    a.n[p] = n;
                    a.b[p] = b;
                    a.v[p] = v;
                }
            }
        }
    }
}

template <int RULE, int ARITH>
cudaError_t launch_direct(const DenseArgs& a, int num_sms, cudaStream_t stream) {
    const int64_t nq = (a.P + 3) / 4;
    int64_t grid = (nq + kDirectThreads - 1) / kDirectThreads;
    if (grid > 8 * (int64_t)num_sms) grid = 8 * (int64_t)num_sms;
    return launch_pdl(fasgd_direct_kernel<RULE, ARITH>, (unsigned)grid, kDirectThreads, 0, stream, a);
}

template <int RULE, int ARITH>
cudaError_t launch_rule(const DenseArgs& a, int num_sms, cudaStream_t stream) {
    if constexpr (RULE != kRuleSgd) {
        if (a.vsum != nullptr) {
            if (a.K != 1) return cudaErrorInvalidValue;
            return launch_ch<RULE, ARITH, 1, true>(a, num_sms, stream);
        }
    }
    if (a.P / kTile < kDirectTilesPerSm * num_sms) return launch_direct<RULE, ARITH>(a, num_sms, stream);
    // Gradient slices per stage: K rounded up to a power of two, at most 8.
    // K > 8 takes several stages per tile: two blocks of 256 consumers per SM
    // keep more stages in flight there (P = 50M, K = 16: 686.8 against
    // 704.0 us per pass); up to K = 8 one block of 512 is faster (226.8
    // against 232.1 us at P = 25M, K = 8).
    if (a.K > 8) return launch_ch<RULE, ARITH, 8, false, 256>(a, num_sms, stream);
    if (a.K > 4) return launch_ch<RULE, ARITH, 8>(a, num_sms, stream);
    if (a.K > 2) return launch_ch<RULE, ARITH, 4>(a, num_sms, stream);
    if (a.K > 1) return launch_ch<RULE, ARITH, 2>(a, num_sms, stream);
    return launch_ch<RULE, ARITH, 1>(a, num_sms, stream);
}

}  // namespace

cudaError_t launch_dense(const DenseArgs& a, int rule, bool exact, int num_sms,
                         cudaStream_t stream, int64_t* launches) {
    const bool ftz = a.sp.eps >= kFtzSafeEps;
    cudaError_t st;
    if (rule == kRuleSgd)
        st = launch_rule<kRuleSgd, kArithApprox>(a, num_sms, stream);  // exact in every mode
    else if (rule == kRuleFasgd)
        st = exact ? launch_rule<kRuleFasgd, kArithExact>(a, num_sms, stream)
             : ftz ? launch_rule<kRuleFasgd, kArithApproxFtz>(a, num_sms, stream)
                   : launch_rule<kRuleFasgd, kArithApprox>(a, num_sms, stream);
    else
        st = exact ? launch_rule<kRuleFasgdStd, kArithExact>(a, num_sms, stream)
             : ftz ? launch_rule<kRuleFasgdStd, kArithApproxFtz>(a, num_sms, stream)
                   : launch_rule<kRuleFasgdStd, kArithApprox>(a, num_sms, stream);
    if (st == cudaSuccess) ++*launches;
    return st;
}

}  // namespace fasgd
