// B-FASGD transmission decisions, per parameter (paper Sec. 2.3, Eq. 9): the
// send (push) or fetch decision and the compaction of the kept entries into
// an ascending index list and the matching values (the push's gradient, or
// the server's theta for a fetch).  Push and fetch draws come from separate
// Philox counter streams (bit 31 of the client word).
//
// Three kernels, all on the caller's stream:
//   1. mask:    per tile of 8192 parameters, draw u_p (Philox4x32-10), take
//               the Eq. 9 decision against v_p, write one bit per parameter
//               and the tile's count of sent entries;
//   2. scan:    exclusive prefix sum of the tile counts (one block) and the
//               total m;
//   3. compact: per tile, rebuild each parameter's rank among the sent ones
//               from the bit mask (warp popc + shuffles, block scan over
//               warps) and write idx[rank] = p, val[rank] = grad[p], staged
//               per warp in shared memory so that the stores are coalesced.
// The order of the output is the order of p, so the result is unique and
// does not depend on the launch; no atomics are used.  Traffic per
// parameter: v (4 B) + grad (4 B) + 2 x 1/8 B of mask, plus 8 B per sent
// entry.  Each lane issues all eight of its 128-bit loads before it computes.

#include "eq9.cuh"
#include "kernels.cuh"
#include "pdl.cuh"

namespace fasgd {
namespace {

constexpr int kWarps = kSelectThreads / 32;
constexpr int kWarpSpan = kSelectTile / kWarps;  // 1024 parameters per warp
constexpr int kIters = kWarpSpan / 128;          // 8 passes of 32 lanes x 4
constexpr unsigned kFull = 0xffffffffu;

// The four values e .. e+3 of x (zero past P; FULL: the tile lies inside P).
template <bool FULL>
__device__ __forceinline__ float4 load_quad(const float* x, int64_t e, int64_t P) {
    if (FULL || e + 3 < P) return __ldcs(reinterpret_cast<const float4*>(x + e));
    float t[4] = {0.f, 0.f, 0.f, 0.f};
    for (int j = 0; j < 4; ++j)
        if (e + j < P) t[j] = x[e + j];
    return make_float4(t[0], t[1], t[2], t[3]);
}

template <bool FULL, bool SCALE_D>
__device__ __forceinline__ void mask_tile(const SelectArgs& a) {
    __shared__ int32_t warp_cnt[kWarps];
    const int lane = threadIdx.x & 31;
    const int warp = threadIdx.x >> 5;
    const int64_t tile_start = (int64_t)blockIdx.x * kSelectTile;
    const int64_t warp_start = tile_start + (int64_t)warp * kWarpSpan;
    // All of this lane's v loads first (eight quads), then the draws.
    float4 v4[kIters];
#pragma unroll
    for (int it = 0; it < kIters; ++it) v4[it] = load_quad<FULL>(a.v, warp_start + it * 128 + 4 * lane, a.P);
    const uint32_t e_lane = (uint32_t)(warp_start + 4 * lane);  // P < 2^31
    int cnt = 0;
#pragma unroll
    for (int it = 0; it < kIters; ++it) {
        const uint32_t e = e_lane + it * 128;
        uint32_t nib = 0;
        if (FULL || e < a.P) {
            const Philox4 r = philox4x32_10(e >> 2, a.client_word, a.push_lo, a.push_hi, a.round_key0, a.round_key1);
            nib = (send_test<SCALE_D>(r.x[0] >> 8, v4[it].x, a.c, a.eps_b) ? 1u : 0u) |
                  (send_test<SCALE_D>(r.x[1] >> 8, v4[it].y, a.c, a.eps_b) ? 2u : 0u) |
                  (send_test<SCALE_D>(r.x[2] >> 8, v4[it].z, a.c, a.eps_b) ? 4u : 0u) |
                  (send_test<SCALE_D>(r.x[3] >> 8, v4[it].w, a.c, a.eps_b) ? 8u : 0u);
            if (!FULL) {
                const int64_t valid = a.P - e;  // parameters past P are never sent
                if (valid < 4) nib &= (1u << valid) - 1u;
            }
        }
        cnt += __popc(nib);
        // Eight lanes' nibbles form one 32-bit mask word (32 consecutive parameters).
        uint32_t w = nib << (4 * (lane & 7));
        w |= __shfl_xor_sync(kFull, w, 1);
        w |= __shfl_xor_sync(kFull, w, 2);
        w |= __shfl_xor_sync(kFull, w, 4);
        if ((lane & 7) == 0)
            a.mask[(warp_start >> 5) + it * 4 + (lane >> 3)] = w;
    }
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) cnt += __shfl_xor_sync(kFull, cnt, off);
    if (lane == 0) warp_cnt[warp] = cnt;
    __syncthreads();
    if (threadIdx.x == 0) {
        int32_t t = 0;
#pragma unroll
        for (int w = 0; w < kWarps; ++w) t += warp_cnt[w];
        a.tile_count[blockIdx.x] = t;
    }
}

// Full tiles (all but perhaps the last) skip the per-quad bounds checks.
// SCALE_D: the form of the Eq. 9 test for this call's c (send_form).
template <bool SCALE_D>
__global__ void __launch_bounds__(kSelectThreads) bfasgd_mask_kernel(const __grid_constant__ SelectArgs a) {
    pdl_wait();
    pdl_trigger();
    if ((int64_t)(blockIdx.x + 1) * kSelectTile <= a.P)
        mask_tile<true, SCALE_D>(a);
    else
        mask_tile<false, SCALE_D>(a);
}

constexpr int kScanThreads = 1024;

__global__ void __launch_bounds__(kScanThreads) bfasgd_scan_kernel(const __grid_constant__ SelectArgs a) {
    __shared__ int64_t warp_sum[kScanThreads / 32];
    pdl_wait();
    pdl_trigger();
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int per = (a.ntiles + kScanThreads - 1) / kScanThreads;
    const int lo = tid * per;
    const int hi = min(lo + per, a.ntiles);
    // Up to four counts per thread (P up to 32M) are loaded at once and kept.
    constexpr int kKeep = 4;
    int32_t kept[kKeep];
    int64_t local = 0;
    if (per <= kKeep) {
#pragma unroll
        for (int k = 0; k < kKeep; ++k) kept[k] = lo + k < hi ? a.tile_count[lo + k] : 0;
#pragma unroll
        for (int k = 0; k < kKeep; ++k) local += kept[k];
    } else {
        for (int t = lo; t < hi; ++t) local += a.tile_count[t];
    }
    // Inclusive scan of the per-thread sums across the block.
    int64_t incl = local;
#pragma unroll
    for (int off = 1; off < 32; off <<= 1) {
        const int64_t y = __shfl_up_sync(kFull, incl, off);
        if (lane >= off) incl += y;
    }
    if (lane == 31) warp_sum[warp] = incl;
    __syncthreads();
    if (warp == 0) {
        int64_t s = warp_sum[lane];
#pragma unroll
        for (int off = 1; off < 32; off <<= 1) {
            const int64_t y = __shfl_up_sync(kFull, s, off);
            if (lane >= off) s += y;
        }
        warp_sum[lane] = s;  // inclusive over warps
    }
    __syncthreads();
    int64_t run = incl - local + (warp > 0 ? warp_sum[warp - 1] : 0);  // exclusive prefix
    if (per <= kKeep) {
#pragma unroll
        for (int k = 0; k < kKeep; ++k)
            if (lo + k < hi) {
                a.tile_base[lo + k] = run;
                run += kept[k];
            }
    } else {
        for (int t = lo; t < hi; ++t) {
            a.tile_base[t] = run;
            run += a.tile_count[t];
        }
    }
    if (tid == kScanThreads - 1) *a.count = warp_sum[kScanThreads / 32 - 1];
}

// Per warp and pass, the kept (index, value) pairs are first put in rank
// order in shared memory, then written to idx and val by consecutive lanes
// (coalesced), instead of each lane storing its own pairs at scattered ranks.
constexpr int kPassParams = 128;

template <bool FULL>
__device__ __forceinline__ void compact_tile(const SelectArgs& a, uint2* stage) {
    __shared__ int32_t warp_cnt[kWarps];
    const int lane = threadIdx.x & 31;
    const int warp = threadIdx.x >> 5;
    const int64_t tile_start = (int64_t)blockIdx.x * kSelectTile;
    const int64_t warp_start = tile_start + (int64_t)warp * kWarpSpan;
    // Lane l holds the mask word of parameters warp_start + 32 l .. + 31.  The
    // word, the tile's output base and the value quads are all loaded before
    // anything waits on them.
    const uint32_t word = a.mask[(warp_start >> 5) + lane];
    const int64_t tile_out = a.tile_base[blockIdx.x];
    float4 g4[kIters];
#pragma unroll
    for (int it = 0; it < kIters; ++it)
        g4[it] = load_quad<FULL>(a.values, warp_start + it * kPassParams + 4 * lane, a.P);
    const int c = __popc(word);
    int incl = c;
#pragma unroll
    for (int off = 1; off < 32; off <<= 1) {
        const int y = __shfl_up_sync(kFull, incl, off);
        if (lane >= off) incl += y;
    }
    const int excl = incl - c;  // rank of this word's first kept entry in the warp's span
    if (lane == 31) warp_cnt[warp] = incl;
    __syncthreads();
    int64_t out = tile_out;
    for (int w = 0; w < warp; ++w) out += warp_cnt[w];
    int32_t* idx_w = a.idx + out;
    float* val_w = a.val + out;
    const int32_t e_lane = (int32_t)(warp_start + 4 * lane);  // P < 2^31
    const int sh = 4 * (lane & 7);
#pragma unroll
    for (int it = 0; it < kIters; ++it) {
        // This lane's quad lies in word (4 it + lane / 8), bits sh .. sh + 3.
        const int owner = it * 4 + (lane >> 3);
        const uint32_t w = __shfl_sync(kFull, word, owner);
        const int wbase = __shfl_sync(kFull, excl, owner);
        const int pass_base = __shfl_sync(kFull, excl, it * 4);
        const int pass_end = __shfl_sync(kFull, incl, it * 4 + 3);
        const uint32_t nib = (w >> sh) & 0xFu;
        int r = wbase - pass_base + __popc(w & ((1u << sh) - 1u));
        const int32_t e = e_lane + it * kPassParams;
        const uint32_t g[4] = {__float_as_uint(g4[it].x), __float_as_uint(g4[it].y),
                               __float_as_uint(g4[it].z), __float_as_uint(g4[it].w)};
#pragma unroll
        for (int j = 0; j < 4; ++j)
            if ((nib >> j) & 1u) stage[r++] = make_uint2((uint32_t)(e + j), g[j]);
        __syncwarp();
        for (int k = lane; k < pass_end - pass_base; k += 32) {
            const uint2 pr = stage[k];
            idx_w[pass_base + k] = (int32_t)pr.x;
            val_w[pass_base + k] = __uint_as_float(pr.y);
        }
        __syncwarp();
    }
}

__global__ void __launch_bounds__(kSelectThreads) bfasgd_compact_kernel(const __grid_constant__ SelectArgs a) {
    __shared__ uint2 stage[kWarps][kPassParams];
    pdl_wait();
    pdl_trigger();
    if ((int64_t)(blockIdx.x + 1) * kSelectTile <= a.P)
        compact_tile<true>(a, stage[threadIdx.x >> 5]);
    else
        compact_tile<false>(a, stage[threadIdx.x >> 5]);
}

}  // namespace

void select_key_schedule(SelectArgs& a, uint64_t seed) {
    philox_key_schedule(seed, a.round_key0, a.round_key1);
}

cudaError_t launch_select(const SelectArgs& a, cudaStream_t stream, int64_t* launches) {
    cudaError_t st = send_form(a.c)
                         ? launch_pdl(bfasgd_mask_kernel<true>, a.ntiles, kSelectThreads, 0, stream, a)
                         : launch_pdl(bfasgd_mask_kernel<false>, a.ntiles, kSelectThreads, 0, stream, a);
    if (st != cudaSuccess) return st;
    ++*launches;
    st = launch_pdl(bfasgd_scan_kernel, 1, kScanThreads, 0, stream, a);
    if (st != cudaSuccess) return st;
    ++*launches;
    st = launch_pdl(bfasgd_compact_kernel, a.ntiles, kSelectThreads, 0, stream, a);
    if (st != cudaSuccess) return st;
    ++*launches;
    return cudaSuccess;
}

}  // namespace fasgd

// ---------------------------------------------------------------------------
// Allocation-free variant of bfasgd_select_compact for callers that may not
// allocate device memory (see include/fasgd.h).  The same three kernels run
// with their scratch in one fixed static device array instead of handle-owned
// buffers.
// ---------------------------------------------------------------------------
#include <cmath>
#include <cstdio>
#include <mutex>

namespace fasgd {
void set_handleless_error(const char* msg);  // defined in runtime.cu
}

namespace {

constexpr int64_t kNoallocTiles = BFASGD_NOALLOC_PMAX / fasgd::kSelectTile;          // 2048
constexpr int64_t kNoallocMaskBytes = kNoallocTiles * fasgd::kSelectTileWords * 4;  // 2 MiB
constexpr int64_t kNoallocCountBytes = kNoallocTiles * 4;
constexpr int64_t kNoallocBaseBytes = kNoallocTiles * 8;
static_assert(kNoallocMaskBytes + kNoallocCountBytes + kNoallocBaseBytes ==
                  BFASGD_NOALLOC_SCRATCH_BYTES,
              "scratch size in fasgd.h out of date");
static_assert(kNoallocMaskBytes % 256 == 0 && kNoallocCountBytes % 8 == 0, "scratch layout");

// Mask words, then int32 tile counts, then int64 tile bases.
static __device__ __align__(256) unsigned char g_noalloc_scratch[BFASGD_NOALLOC_SCRATCH_BYTES];

constexpr int kMaxDevices = 64;
std::mutex g_noalloc_mutex;
void* g_noalloc_addr[kMaxDevices] = {};

// Device address of the static scratch on the current device, looked up once
// per device.  Host code cannot use the symbol itself as a device pointer.
// The look-up is a runtime call that does not belong in a stream capture:
// if it is still to be made while `stream` is capturing, *capturing is set
// and nothing is done.
cudaError_t noalloc_scratch(cudaStream_t stream, unsigned char** out, bool* capturing) {
    *capturing = false;
    int dev = 0;
    cudaError_t st = cudaGetDevice(&dev);
    if (st != cudaSuccess) return st;
    if (dev < 0 || dev >= kMaxDevices) return cudaErrorInvalidDevice;
    std::lock_guard<std::mutex> lock(g_noalloc_mutex);
    if (g_noalloc_addr[dev] == nullptr) {
        cudaStreamCaptureStatus cs = cudaStreamCaptureStatusNone;
        st = cudaStreamIsCapturing(stream, &cs);
        if (st != cudaSuccess) return st;
        if (cs != cudaStreamCaptureStatusNone) {
            *capturing = true;
            return cudaSuccess;
        }
        void* p = nullptr;
        st = cudaGetSymbolAddress(&p, g_noalloc_scratch);
        if (st != cudaSuccess) return st;
        g_noalloc_addr[dev] = p;
    }
    *out = static_cast<unsigned char*>(g_noalloc_addr[dev]);
    return cudaSuccess;
}

bool aligned_to(const void* p, uintptr_t a) {
    return (reinterpret_cast<uintptr_t>(p) & (a - 1)) == 0;
}

int noalloc_fail(int code, const char* msg) {
    fasgd::set_handleless_error(msg);
    return code;
}

}  // namespace

extern "C" int bfasgd_select_compact_noalloc(int64_t P, const float* grad, const float* v,
                                             float c, float eps_b, uint64_t seed, int32_t client,
                                             uint64_t push_no, int32_t* idx, float* val,
                                             int64_t* n_dev, void* stream) {
    if (P < 1 || P > BFASGD_NOALLOC_PMAX) {
        char buf[160];
        snprintf(buf, sizeof buf,
                 "bfasgd_select_compact_noalloc: P=%lld outside [1, %lld], the size of its "
                 "static scratch", (long long)P, (long long)BFASGD_NOALLOC_PMAX);
        return noalloc_fail(FASGD_EINVAL, buf);
    }
    if (client < 0) return noalloc_fail(FASGD_EINVAL, "bfasgd_select_compact_noalloc: client < 0");
    if (grad == nullptr || v == nullptr || !aligned_to(grad, 16) || !aligned_to(v, 16))
        return noalloc_fail(FASGD_EINVAL,
                            "bfasgd_select_compact_noalloc: grad and v must be non-NULL "
                            "16-byte aligned device pointers");
    if (idx == nullptr || val == nullptr || n_dev == nullptr || !aligned_to(idx, 4) ||
        !aligned_to(val, 4) || !aligned_to(n_dev, 8))
        return noalloc_fail(FASGD_EINVAL,
                            "bfasgd_select_compact_noalloc: idx, val, n_dev must be non-NULL "
                            "and aligned");
    if (!(c >= 0.f) || !(eps_b >= 0.f) || !std::isfinite(eps_b))
        return noalloc_fail(FASGD_EINVAL,
                            "bfasgd_select_compact_noalloc: need c >= 0 and finite eps_b >= 0");
    unsigned char* scratch = nullptr;
    bool capturing = false;
    cudaError_t st = noalloc_scratch(static_cast<cudaStream_t>(stream), &scratch, &capturing);
    if (st != cudaSuccess)
        return noalloc_fail(FASGD_ECUDA, "bfasgd_select_compact_noalloc: cannot address the "
                                         "static scratch on this device");
    if (capturing)
        return noalloc_fail(FASGD_EINVAL,
                            "bfasgd_select_compact_noalloc: the first call on a device looks up "
                            "its static scratch and must come before any stream capture");
    fasgd::SelectArgs a;
    a.values = grad;
    a.v = v;
    a.idx = idx;
    a.val = val;
    a.count = n_dev;
    a.mask = reinterpret_cast<uint32_t*>(scratch);
    a.tile_count = reinterpret_cast<int32_t*>(scratch + kNoallocMaskBytes);
    a.tile_base = reinterpret_cast<int64_t*>(scratch + kNoallocMaskBytes + kNoallocCountBytes);
    a.P = P;
    a.ntiles = fasgd::select_tiles(P);
    a.c = c;
    a.eps_b = eps_b;
    fasgd::select_key_schedule(a, seed);
    a.client_word = (uint32_t)client;
    a.push_lo = (uint32_t)push_no;
    a.push_hi = (uint32_t)(push_no >> 32);
    int64_t launches = 0;
    st = fasgd::launch_select(a, static_cast<cudaStream_t>(stream), &launches);
    if (st != cudaSuccess)
        return noalloc_fail(FASGD_ECUDA, cudaGetErrorString(st));
    return FASGD_OK;
}
