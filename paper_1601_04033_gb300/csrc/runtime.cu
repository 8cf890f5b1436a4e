// Host runtime behind include/fasgd.h: the handle, argument checks, the
// queue of pending pushes, the per-push staleness factors and the launches.
//
// Protocol (paper Sec. 2.1): a client push carries its gradient and the
// timestamp j of the parameters it was computed on; the server applies
// pushes one at a time in arrival order, each at the server timestamp T it
// finds (step-staleness tau = T - j), and T grows by one per applied push.
// Here a batch of K queued pushes is applied by one call: push k of the
// batch sees T + k.  The per-push factor alpha(tau) = alpha / max(tau, 1)
// (Eq. 1, Eq. 7 without the per-element v) is formed on the host in fp64 and
// rounded once to fp32.

#include <cuda_runtime.h>
#include <nvtx3/nvToolsExt.h>

#include <cmath>
#include <cstdarg>
#include <cstdio>
#include <cstring>
#include <deque>
#include <new>
#include <string>
#include <vector>

#include "eq9.cuh"
#include "fasgd.h"
#include "kernels.cuh"
#include "message.cuh"
#include "tensors.cuh"

namespace {

constexpr int64_t kMaxQueue = int64_t(1) << 20;
constexpr int32_t kMaxLambda = int32_t(1) << 20;

thread_local std::string g_create_error;

enum PushKind { kDense = 0, kSparse = 1, kMessage = 2, kBudget = 3 };

struct Push {
    int kind;              // PushKind
    int32_t client;
    int64_t j;
    const float* grad;     // dense
    const int32_t* idx;    // sparse
    const float* val;
    const int64_t* n_dev;
    int64_t n_max;
    int stage;             // staging slot of a host push, -1 otherwise
    int32_t* flag;         // message push: where to report the decision (may be null)
    int64_t budget;        // budget push: expected parameters per push
    uint8_t* sent_out;     // budget push: caller copies of the decisions (each may be null)
    float* c_out;
    int64_t* count_out;
};

// An NVTX range around a call that launches work or copies (visible to
// Nsight tools and to ncu --nvtx; free when no tool is attached).
struct TraceRange {
    explicit TraceRange(const char* name) { nvtxRangePushA(name); }
    ~TraceRange() { nvtxRangePop(); }
    TraceRange(const TraceRange&) = delete;
    TraceRange& operator=(const TraceRange&) = delete;
};

bool aligned(const void* p, uintptr_t a) { return (reinterpret_cast<uintptr_t>(p) & (a - 1)) == 0; }

std::string vformat(const char* fmt, va_list ap) {
    char buf[512];
    vsnprintf(buf, sizeof buf, fmt, ap);
    return buf;
}

// Makes h's device current for the lifetime of the guard.
struct DeviceGuard {
    int prev = -1;
    explicit DeviceGuard(int dev) {
        if (cudaGetDevice(&prev) == cudaSuccess && prev != dev) cudaSetDevice(dev);
        else prev = -1;
    }
    ~DeviceGuard() {
        if (prev >= 0) cudaSetDevice(prev);
    }
};

}  // namespace

namespace fasgd {
// Records the failure of a call made without a handle (read back through
// fasgd_last_error(NULL)).
void set_handleless_error(const char* msg) { g_create_error = msg; }
}  // namespace fasgd

struct fasgd_s {
    int64_t P = 0;
    int32_t lambda = 0;
    float alpha = 0.f;
    int32_t variant = FASGD_FASGD;
    float gamma = 0.95f, beta = 0.95f, eps = 1e-4f, c_push = 0.f, eps_b = 1e-8f;
    float c_fetch = 0.f;
    bool exact = false;     // exact fp32 arithmetic instead of the fast forms
    uint64_t seed = 0;
    cudaStream_t stream = nullptr;
    int device = 0;
    int num_sms = 0;
    float* theta = nullptr;
    float* n = nullptr;
    float* b = nullptr;
    float* v = nullptr;
    uint32_t* mask = nullptr;
    int32_t* tile_count = nullptr;
    int64_t* tile_base = nullptr;
    int32_t* dev_err = nullptr;
    int32_t ntiles = 0;
    // Host pushes: device staging slots filled on copy_stream, so the copies
    // of the next pushes overlap the pass that consumes the previous ones.
    std::vector<float*> stage;
    std::vector<char> stage_busy;       // held by a queued push
    std::vector<char> stage_used;       // slot_free has been recorded
    std::vector<uint64_t> stage_seq;    // pass that last read the slot (larger = later)
    uint64_t pass_seq = 0;
    std::vector<cudaEvent_t> slot_ready;  // the copy into the slot is done
    std::vector<cudaEvent_t> slot_free;   // the last pass reading the slot is done
    cudaStream_t copy_stream = nullptr;
    cudaStream_t pull_stream = nullptr;   // pulls run beside the next host copies
    cudaEvent_t order_ev = nullptr;
    cudaEvent_t pull_done_ev = nullptr;
    cudaEvent_t switch_ev = nullptr;      // orders a new stream after the previous one
    std::deque<Push> fifo;
    int64_t T = 0;
    int64_t launches = 0;
    // Test hook (fasgd_selftest_fail_pass): the pass of fasgd_apply_pending
    // this many passes from now reports a launch failure instead of running;
    // -1: off.
    int32_t fail_pass_in = -1;
    // True when the next pass is the one to fail (the countdown advances).
    bool injected_failure() {
        if (fail_pass_in < 0) return false;
        if (fail_pass_in-- > 0) return false;
        return true;
    }
    std::vector<uint64_t> push_count;
    std::vector<uint64_t> fetch_count;
    std::string err;

    int fail(int code, const char* fmt, ...) {
        va_list ap;
        va_start(ap, fmt);
        err = vformat(fmt, ap);
        va_end(ap);
        return code;
    }
    int cuda_fail(cudaError_t st, const char* what) {
        return fail(st == cudaErrorMemoryAllocation ? FASGD_ENOMEM : FASGD_ECUDA, "%s: %s", what,
                    cudaGetErrorString(st));
    }
    // Per-message B-FASGD: the gradient cache (lambda slots of cache_stride
    // floats, allocated by the first message push) and the partial sums.
    float* grad_cache = nullptr;
    int64_t cache_stride = 0;
    float2* msg_partial = nullptr;
    float2* msg_chunks = nullptr;   // chunk sums of v (128 parameters each)
    bool msg_sums_valid = false;    // msg_chunks holds those of the current v

    // Per-tensor B-FASGD: the partition, its work items on the device, the
    // item sums of v and the decision of the latest call.
    std::vector<int64_t> tensor_sizes;
    fasgd::TensorItem* t_items = nullptr;
    int32_t t_nitems = 0;
    int32_t* t_item_begin = nullptr;
    int32_t* t_sizes = nullptr;
    float2* t_partial = nullptr;
    uint8_t* t_sent = nullptr;
    float* t_c = nullptr;
    int64_t* t_count = nullptr;
    float* t_vbar = nullptr;       // cached tensor means
    uint8_t* t_dirty = nullptr;    // tensors whose v changed since their mean was formed
    long long* t_cprev = nullptr;  // last threshold per stream (push, fetch)
    bool t_sums_valid = false;   // t_partial holds the item sums of the current v

    void free_tensors() {
        cudaFree(t_items);
        cudaFree(t_item_begin);
        cudaFree(t_sizes);
        cudaFree(t_partial);
        cudaFree(t_sent);
        cudaFree(t_c);
        cudaFree(t_count);
        cudaFree(t_vbar);
        cudaFree(t_dirty);
        cudaFree(t_cprev);
        t_vbar = nullptr;
        t_dirty = nullptr;
        t_cprev = nullptr;
        t_items = nullptr;
        t_item_begin = nullptr;
        t_sizes = nullptr;
        t_partial = nullptr;
        t_sent = nullptr;
        t_c = nullptr;
        t_count = nullptr;
        t_nitems = 0;
        t_sums_valid = false;
        tensor_sizes.clear();
    }

    // One per-tensor decision of `stream_id` for `client` under `budget`
    // (advancing the client's counter); the decisions land in t_sent.
    cudaError_t launch_budget(uint32_t stream_id, int32_t client, int64_t budget,
                              uint8_t* sent_out, float* c_out, int64_t* count_out,
                              std::vector<uint64_t>& counter) {
        fasgd::TensorArgs a;
        std::memset(&a, 0, sizeof a);
        a.v = v;
        a.items = t_items;
        a.n_items = t_nitems;
        a.item_begin = t_item_begin;
        a.sizes = t_sizes;
        a.T = (int32_t)tensor_sizes.size();
        a.partial = t_partial;
        a.eps_b = eps_b;
        const int64_t B = budget < P ? budget : P;
        a.limit = B * (int64_t(1) << 32);
        fasgd::philox_key_schedule(seed, a.round_key0, a.round_key1);
        const uint64_t n = counter[(size_t)client];
        a.client_word = (uint32_t)client | (stream_id << 31);
        a.n_lo = (uint32_t)n;
        a.n_hi = (uint32_t)(n >> 32);
        a.sent = t_sent;
        a.c_out = t_c;
        a.count_out = t_count;
        a.user_sent = sent_out;
        a.user_c = c_out;
        a.user_count = count_out;
        a.vbar_cache = t_vbar;
        a.dirty = t_dirty;
        a.c_prev = t_cprev + stream_id;
        a.all_dirty = t_sums_valid ? 0 : 1;
        a.mark_dirty = (stream_id == 0 && variant != FASGD_ASGD && variant != FASGD_SASGD) ? 1 : 0;
        cudaError_t st = fasgd::launch_tensor_decide(a, t_sums_valid, stream, &launches);
        if (st == cudaSuccess) {
            t_sums_valid = true;
            counter[(size_t)client] = n + 1;
        }
        return st;
    }
    fasgd::RangeArgs range_args() const {
        fasgd::RangeArgs r;
        std::memset(&r, 0, sizeof r);
        r.theta = theta;
        r.n = n;
        r.b = b;
        r.v = v;
        r.sp = stat_params();
        r.items = t_items;
        r.n_items = t_nitems;
        r.sent = t_sent;
        r.partial = t_partial;
        return r;
    }

    cudaError_t ensure_message_scratch(bool cache) {
        cudaError_t st = cudaSuccess;
        if (msg_partial == nullptr)
            st = cudaMalloc(reinterpret_cast<void**>(&msg_partial),
                            fasgd::kMessageMaxBlocks * sizeof(float2));
        if (st == cudaSuccess && msg_chunks == nullptr) {
            st = cudaMalloc(reinterpret_cast<void**>(&msg_chunks),
                            (size_t)((P + fasgd::kVsumChunk - 1) / fasgd::kVsumChunk) * sizeof(float2));
            msg_sums_valid = false;
        }
        if (st == cudaSuccess && cache && grad_cache == nullptr) {
            cache_stride = (P + 63) / 64 * 64;   // 256-byte aligned slots
            const size_t bytes = (size_t)lambda * (size_t)cache_stride * sizeof(float);
            st = cudaMalloc(reinterpret_cast<void**>(&grad_cache), bytes);
            if (st == cudaSuccess) st = cudaMemsetAsync(grad_cache, 0, bytes, stream);
            if (st != cudaSuccess && grad_cache != nullptr) {
                cudaFree(grad_cache);
                grad_cache = nullptr;
            }
        }
        return st;
    }

    // Arguments of one per-message decision of `stream_id` for `client`, its
    // n-th message of that stream, copying src -> dst if transmitted.
    fasgd::MessageArgs message_args(uint32_t stream_id, int32_t client, const float* src,
                                    float* dst, int32_t* flag, float c, uint64_t n,
                                    float* vbar_out) const {
        fasgd::MessageArgs a;
        std::memset(&a, 0, sizeof a);
        a.v = v;
        a.P = P;
        a.partial = msg_partial;
        a.nblocks = fasgd::message_partial_blocks(P);
        a.chunks = msg_chunks;
        a.from_v = msg_sums_valid ? 0 : 1;
        a.c = c;
        a.eps_b = eps_b;
        fasgd::philox_key_schedule(seed, a.round_key0, a.round_key1);
        a.client_word = (uint32_t)client | (stream_id << 31);
        a.n_lo = (uint32_t)n;
        a.n_hi = (uint32_t)(n >> 32);
        a.src = src;
        a.dst = dst;
        a.flag_out = flag;
        a.vbar_out = vbar_out;
        return a;
    }

    // One per-message decision of `stream_id` for `client` (advancing its
    // counter), copying src -> dst if transmitted.
    cudaError_t launch_message(uint32_t stream_id, int32_t client, const float* src, float* dst,
                               int32_t* flag, float c, std::vector<uint64_t>* counter,
                               float* vbar_out = nullptr) {
        const uint64_t n = counter != nullptr ? (*counter)[(size_t)client] : 0;
        const fasgd::MessageArgs a = message_args(stream_id, client, src, dst, flag, c, n, vbar_out);
        cudaError_t st = fasgd::launch_message(a, num_sms, stream, &launches);
        if (st == cudaSuccess) {
            msg_sums_valid = true;
            if (counter != nullptr) (*counter)[(size_t)client] = n + 1;
        }
        return st;
    }

    // Streams and events for host copies and pulls, created on first use.
    cudaError_t ensure_aux() {
        cudaError_t st = cudaSuccess;
        if (copy_stream == nullptr)
            st = cudaStreamCreateWithFlags(&copy_stream, cudaStreamNonBlocking);
        if (st == cudaSuccess && pull_stream == nullptr)
            st = cudaStreamCreateWithFlags(&pull_stream, cudaStreamNonBlocking);
        if (st == cudaSuccess && order_ev == nullptr)
            st = cudaEventCreateWithFlags(&order_ev, cudaEventDisableTiming);
        if (st == cudaSuccess && pull_done_ev == nullptr)
            st = cudaEventCreateWithFlags(&pull_done_ev, cudaEventDisableTiming);
        return st;
    }
    fasgd::StatParams stat_params() const {
        fasgd::StatParams sp;
        sp.gamma = gamma;
        sp.one_m_gamma = 1.0f - gamma;
        sp.beta = beta;
        sp.one_m_beta = 1.0f - beta;
        sp.eps = eps;
        return sp;
    }
    // alpha(tau) of Eq. 1 / Eq. 7 (the v factor of Eq. 7 is per element).
    float coef(int64_t tau) const {
        if (variant == FASGD_ASGD) return alpha;
        const int64_t t = tau < 1 ? 1 : tau;
        return (float)((double)alpha / (double)t);
    }
    void free_all() {
        float* arrs[] = {theta, n, b, v};
        for (float* p : arrs) cudaFree(p);
        cudaFree(mask);
        cudaFree(tile_count);
        cudaFree(tile_base);
        cudaFree(dev_err);
        cudaFree(grad_cache);
        cudaFree(msg_partial);
        cudaFree(msg_chunks);
        msg_chunks = nullptr;
        msg_sums_valid = false;
        grad_cache = nullptr;
        msg_partial = nullptr;
        free_tensors();
        for (float* s : stage) cudaFree(s);
        for (cudaEvent_t e : slot_ready) cudaEventDestroy(e);
        for (cudaEvent_t e : slot_free) cudaEventDestroy(e);
        slot_ready.clear();
        slot_free.clear();
        if (order_ev) cudaEventDestroy(order_ev);
        if (pull_done_ev) cudaEventDestroy(pull_done_ev);
        if (switch_ev) cudaEventDestroy(switch_ev);
        switch_ev = nullptr;
        if (copy_stream) cudaStreamDestroy(copy_stream);
        if (pull_stream) cudaStreamDestroy(pull_stream);
        order_ev = pull_done_ev = nullptr;
        copy_stream = pull_stream = nullptr;
        theta = n = b = v = nullptr;
        mask = nullptr;
        tile_count = nullptr;
        tile_base = nullptr;
        dev_err = nullptr;
        stage.clear();
    }
};

extern "C" {

int fasgd_create(fasgd_t** h, int64_t P, int32_t lambda, float alpha, int32_t variant) {
    if (h == nullptr) {
        g_create_error = "fasgd_create: h is NULL";
        return FASGD_EINVAL;
    }
    *h = nullptr;
    if (P < 1 || P > FASGD_PMAX) {
        g_create_error = "fasgd_create: P must be in [1, 2^31)";
        return FASGD_EINVAL;
    }
    if (lambda < 1 || lambda > kMaxLambda) {
        g_create_error = "fasgd_create: lambda must be in [1, 2^20]";
        return FASGD_EINVAL;
    }
    if (!std::isfinite(alpha)) {
        g_create_error = "fasgd_create: alpha must be finite";
        return FASGD_EINVAL;
    }
    if (variant != FASGD_ASGD && variant != FASGD_SASGD && variant != FASGD_FASGD &&
        variant != FASGD_FASGD_STD) {
        g_create_error = "fasgd_create: unknown variant";
        return FASGD_EINVAL;
    }
    fasgd_s* s = new (std::nothrow) fasgd_s();
    if (s == nullptr) {
        g_create_error = "fasgd_create: out of host memory";
        return FASGD_ENOMEM;
    }
    s->P = P;
    s->lambda = lambda;
    s->alpha = alpha;
    s->variant = variant;
    s->push_count.assign((size_t)lambda, 0);
    s->fetch_count.assign((size_t)lambda, 0);
    s->ntiles = fasgd::select_tiles(P);
    cudaError_t st = cudaGetDevice(&s->device);
    if (st == cudaSuccess)
        st = cudaDeviceGetAttribute(&s->num_sms, cudaDevAttrMultiProcessorCount, s->device);
    const size_t bytes = (size_t)P * sizeof(float);
    float** arrs[] = {&s->theta, &s->n, &s->b, &s->v};
    for (float** a : arrs)
        if (st == cudaSuccess) st = cudaMalloc(reinterpret_cast<void**>(a), bytes);
    if (st == cudaSuccess)
        st = cudaMalloc(reinterpret_cast<void**>(&s->mask),
                        (size_t)s->ntiles * fasgd::kSelectTileWords * sizeof(uint32_t));
    if (st == cudaSuccess)
        st = cudaMalloc(reinterpret_cast<void**>(&s->tile_count), (size_t)s->ntiles * sizeof(int32_t));
    if (st == cudaSuccess)
        st = cudaMalloc(reinterpret_cast<void**>(&s->tile_base), (size_t)s->ntiles * sizeof(int64_t));
    if (st == cudaSuccess) st = cudaMalloc(reinterpret_cast<void**>(&s->dev_err), sizeof(int32_t));
    for (float** a : arrs)
        if (st == cudaSuccess) st = cudaMemset(*a, 0, bytes);
    if (st == cudaSuccess) st = cudaMemset(s->dev_err, 0, sizeof(int32_t));
    if (st == cudaSuccess) st = cudaDeviceSynchronize();
    if (st != cudaSuccess) {
        g_create_error = std::string("fasgd_create: ") + cudaGetErrorString(st);
        s->free_all();
        delete s;
        return st == cudaErrorMemoryAllocation ? FASGD_ENOMEM : FASGD_ECUDA;
    }
    *h = s;
    return FASGD_OK;
}

void fasgd_destroy(fasgd_t* h) {
    if (h == nullptr) return;
    DeviceGuard g(h->device);
    cudaStreamSynchronize(h->stream);
    if (h->copy_stream) cudaStreamSynchronize(h->copy_stream);
    if (h->pull_stream) cudaStreamSynchronize(h->pull_stream);
    h->free_all();
    delete h;
}

int fasgd_set_hparams(fasgd_t* h, float gamma, float beta, float eps, float c_push, float eps_b,
                      uint64_t seed) {
    if (h == nullptr) return FASGD_EINVAL;
    if (!(gamma >= 0.f && gamma <= 1.f)) return h->fail(FASGD_EINVAL, "gamma must be in [0, 1]");
    if (!(beta >= 0.f && beta < 1.f)) return h->fail(FASGD_EINVAL, "beta must be in [0, 1)");
    if (!(eps >= 0.f) || !std::isfinite(eps)) return h->fail(FASGD_EINVAL, "eps must be finite and >= 0");
    if (!(c_push >= 0.f)) return h->fail(FASGD_EINVAL, "c_push must be >= 0 (may be +inf)");
    if (!(eps_b >= 0.f) || !std::isfinite(eps_b))
        return h->fail(FASGD_EINVAL, "eps_b must be finite and >= 0");
    if (!h->fifo.empty()) return h->fail(FASGD_EAGAIN, "pushes are pending");
    h->gamma = gamma;
    h->beta = beta;
    h->eps = eps;
    h->c_push = c_push;
    h->eps_b = eps_b;
    h->seed = seed;
    return FASGD_OK;
}

int fasgd_set_exact(fasgd_t* h, int32_t exact) {
    if (h == nullptr) return FASGD_EINVAL;
    if (!h->fifo.empty()) return h->fail(FASGD_EAGAIN, "pushes are pending");
    h->exact = exact != 0;
    return FASGD_OK;
}

int fasgd_set_stream(fasgd_t* h, void* stream) {
    if (h == nullptr) return FASGD_EINVAL;
    if (!h->fifo.empty()) return h->fail(FASGD_EAGAIN, "pushes are pending");
    const cudaStream_t s = static_cast<cudaStream_t>(stream);
    if (s == h->stream) return FASGD_OK;
    // What the handle enqueued on the previous stream (passes, selects,
    // copies, pulls) comes before anything it enqueues on the new one.
    DeviceGuard g(h->device);
    cudaError_t st = cudaSuccess;
    if (h->switch_ev == nullptr) st = cudaEventCreateWithFlags(&h->switch_ev, cudaEventDisableTiming);
    if (st == cudaSuccess) st = cudaEventRecord(h->switch_ev, h->stream);
    if (st == cudaSuccess) st = cudaStreamWaitEvent(s, h->switch_ev, 0);
    if (st != cudaSuccess) return h->cuda_fail(st, "fasgd_set_stream");
    h->stream = s;
    return FASGD_OK;
}

int fasgd_set_params(fasgd_t* h, const float* theta0) {
    if (h == nullptr) return FASGD_EINVAL;
    if (theta0 == nullptr) return h->fail(FASGD_EINVAL, "theta0 is NULL");
    if (!h->fifo.empty()) return h->fail(FASGD_EAGAIN, "pushes are pending");
    DeviceGuard g(h->device);
    cudaError_t st = cudaMemcpyAsync(h->theta, theta0, (size_t)h->P * sizeof(float),
                                     cudaMemcpyDefault, h->stream);
    if (st != cudaSuccess) return h->cuda_fail(st, "fasgd_set_params");
    return FASGD_OK;
}

static int check_push(fasgd_t* h, int32_t client, int64_t timestamp) {
    if (client < 0 || client >= h->lambda)
        return h->fail(FASGD_ERANGE, "client %d outside [0, %d)", client, h->lambda);
    if (timestamp < 0 || timestamp > h->T)
        return h->fail(FASGD_ERANGE, "timestamp %lld outside [0, T=%lld]", (long long)timestamp,
                       (long long)h->T);
    if ((int64_t)h->fifo.size() >= kMaxQueue) return h->fail(FASGD_EAGAIN, "push queue is full");
    return FASGD_OK;
}

int fasgd_push(fasgd_t* h, int32_t client, int64_t timestamp, const float* grad) {
    if (h == nullptr) return FASGD_EINVAL;
    if (grad == nullptr || !aligned(grad, 16))
        return h->fail(FASGD_EINVAL, "grad must be a non-NULL 16-byte aligned device pointer");
    int rc = check_push(h, client, timestamp);
    if (rc != FASGD_OK) return rc;
    h->fifo.push_back(Push{kDense, client, timestamp, grad, nullptr, nullptr, nullptr, 0, -1, nullptr});
    return FASGD_OK;
}

int fasgd_push_host(fasgd_t* h, int32_t client, int64_t timestamp, const float* grad_host) {
    TraceRange trace("fasgd_push_host");
    if (h == nullptr) return FASGD_EINVAL;
    if (grad_host == nullptr) return h->fail(FASGD_EINVAL, "grad_host is NULL");
    int rc = check_push(h, client, timestamp);
    if (rc != FASGD_OK) return rc;
    DeviceGuard g(h->device);
    cudaError_t st = h->ensure_aux();
    if (st != cudaSuccess) return h->cuda_fail(st, "fasgd_push_host: streams");
    // Prefer a free slot no pass is still reading; else grow the pool; else
    // take any free slot (its copy then waits for the pass that read it).
    // If no slot is free, the one read longest ago is taken: its reader is the
    // likeliest to have finished, so the copy engine rarely waits on a pass.
    int slot = -1, waiting = -1;
    bool must_wait = false;   // the slot's last reader may still be running
    for (size_t s = 0; s < h->stage.size(); ++s) {
        if (h->stage_busy[s]) continue;
        if (!h->stage_used[s] || cudaEventQuery(h->slot_free[s]) == cudaSuccess) {
            slot = (int)s;
            break;
        }
        if (waiting < 0 || h->stage_seq[s] < h->stage_seq[(size_t)waiting]) waiting = (int)s;
    }
    if (slot < 0 && (int)h->stage.size() < FASGD_KMAX) {
        float* p = nullptr;
        cudaEvent_t ready = nullptr, freed = nullptr;
        st = cudaMalloc(reinterpret_cast<void**>(&p), (size_t)h->P * sizeof(float));
        if (st == cudaSuccess) st = cudaEventCreateWithFlags(&ready, cudaEventDisableTiming);
        if (st == cudaSuccess) st = cudaEventCreateWithFlags(&freed, cudaEventDisableTiming);
        if (st != cudaSuccess) {
            cudaFree(p);
            if (ready) cudaEventDestroy(ready);
            return h->cuda_fail(st, "fasgd_push_host: staging slot");
        }
        h->stage.push_back(p);
        h->stage_busy.push_back(0);
        h->stage_used.push_back(0);
        h->stage_seq.push_back(0);
        h->slot_ready.push_back(ready);
        h->slot_free.push_back(freed);
        slot = (int)h->stage.size() - 1;
    }
    if (slot < 0 && waiting >= 0) {
        slot = waiting;
        must_wait = true;
    }
    if (slot < 0) return h->fail(FASGD_EAGAIN, "%d host pushes already pending", FASGD_KMAX);
    // A slot whose last reader has finished needs no dependency: skipping the
    // wait keeps the copy engine streaming from one copy into the next.
    if (must_wait) st = cudaStreamWaitEvent(h->copy_stream, h->slot_free[(size_t)slot], 0);
    if (st == cudaSuccess)
        st = cudaMemcpyAsync(h->stage[(size_t)slot], grad_host, (size_t)h->P * sizeof(float),
                             cudaMemcpyDefault, h->copy_stream);
    if (st == cudaSuccess) st = cudaEventRecord(h->slot_ready[(size_t)slot], h->copy_stream);
    if (st != cudaSuccess) return h->cuda_fail(st, "fasgd_push_host: copy");
    h->stage_busy[(size_t)slot] = 1;
    h->fifo.push_back(Push{kDense, client, timestamp, h->stage[(size_t)slot], nullptr, nullptr, nullptr, 0, slot, nullptr});
    return FASGD_OK;
}

int bfasgd_push_message(fasgd_t* h, int32_t client, int64_t timestamp, const float* grad,
                        int32_t* sent_dev) {
    if (h == nullptr) return FASGD_EINVAL;
    if (grad == nullptr || !aligned(grad, 16))
        return h->fail(FASGD_EINVAL, "grad must be a non-NULL 16-byte aligned device pointer");
    if (!aligned(sent_dev, 4)) return h->fail(FASGD_EINVAL, "sent_dev must be 4-byte aligned");
    int rc = check_push(h, client, timestamp);
    if (rc != FASGD_OK) return rc;
    DeviceGuard g(h->device);
    cudaError_t st = h->ensure_message_scratch(true);
    if (st != cudaSuccess) return h->cuda_fail(st, "bfasgd_push_message: gradient cache");
    h->fifo.push_back(Push{kMessage, client, timestamp, grad, nullptr, nullptr, nullptr, 0, -1, sent_dev});
    return FASGD_OK;
}

int bfasgd_fetch_message(fasgd_t* h, int32_t client, float* theta_client, int32_t* fetched_dev) {
    TraceRange trace("bfasgd_fetch_message");
    if (h == nullptr) return FASGD_EINVAL;
    if (client < 0 || client >= h->lambda)
        return h->fail(FASGD_ERANGE, "client %d outside [0, %d)", client, h->lambda);
    if (theta_client == nullptr || !aligned(theta_client, 16) || !aligned(fetched_dev, 4))
        return h->fail(FASGD_EINVAL, "theta_client must be a non-NULL 16-byte aligned device "
                                     "pointer (fetched_dev 4-byte aligned)");
    DeviceGuard g(h->device);
    cudaError_t st = h->ensure_message_scratch(false);
    if (st == cudaSuccess)
        st = h->launch_message(1, client, h->theta, theta_client, fetched_dev, h->c_fetch,
                               &h->fetch_count);
    if (st != cudaSuccess) return h->cuda_fail(st, "bfasgd_fetch_message");
    return FASGD_OK;
}

int bfasgd_set_tensors(fasgd_t* h, int32_t T, const int64_t* sizes) {
    TraceRange trace("bfasgd_set_tensors");
    if (h == nullptr) return FASGD_EINVAL;
    if (T < 1 || T > BFASGD_TMAX || sizes == nullptr)
        return h->fail(FASGD_EINVAL, "T must be in [1, %d] and sizes non-NULL", BFASGD_TMAX);
    int64_t total = 0;
    for (int32_t t = 0; t < T; ++t) {
        if (sizes[t] < 1 || sizes[t] > h->P)
            return h->fail(FASGD_EINVAL, "tensor %d has size %lld", t, (long long)sizes[t]);
        total += sizes[t];
        if (total > h->P) break;
    }
    if (total != h->P) return h->fail(FASGD_EINVAL, "tensor sizes do not sum to P");
    if (!h->fifo.empty()) return h->fail(FASGD_EAGAIN, "pushes are pending");
    DeviceGuard g(h->device);
    // Work items: each tensor cut into pieces of at most `chunk` parameters.
    const int64_t chunk = fasgd::tensor_chunk(h->P);
    std::vector<fasgd::TensorItem> items;
    std::vector<int32_t> begin((size_t)T + 1), sz((size_t)T);
    int64_t off = 0;
    for (int32_t t = 0; t < T; ++t) {
        begin[(size_t)t] = (int32_t)items.size();
        sz[(size_t)t] = (int32_t)sizes[t];
        for (int64_t s = 0; s < sizes[t]; s += chunk) {
            const int64_t len = sizes[t] - s < chunk ? sizes[t] - s : chunk;
            items.push_back(fasgd::TensorItem{off + s, (int32_t)len, t});
        }
        off += sizes[t];
    }
    begin[(size_t)T] = (int32_t)items.size();
    cudaError_t st = cudaStreamSynchronize(h->stream);   // no decision still reads the old tables
    h->free_tensors();
    const size_t ni = items.size();
    if (st == cudaSuccess) st = cudaMalloc(reinterpret_cast<void**>(&h->t_items), ni * sizeof(fasgd::TensorItem));
    if (st == cudaSuccess) st = cudaMalloc(reinterpret_cast<void**>(&h->t_item_begin), begin.size() * sizeof(int32_t));
    if (st == cudaSuccess) st = cudaMalloc(reinterpret_cast<void**>(&h->t_sizes), sz.size() * sizeof(int32_t));
    if (st == cudaSuccess) st = cudaMalloc(reinterpret_cast<void**>(&h->t_partial), ni * sizeof(float2));
    if (st == cudaSuccess) st = cudaMalloc(reinterpret_cast<void**>(&h->t_sent), (size_t)T);
    if (st == cudaSuccess) st = cudaMalloc(reinterpret_cast<void**>(&h->t_c), sizeof(float));
    if (st == cudaSuccess) st = cudaMalloc(reinterpret_cast<void**>(&h->t_count), sizeof(int64_t));
    if (st == cudaSuccess) st = cudaMalloc(reinterpret_cast<void**>(&h->t_vbar), (size_t)T * sizeof(float));
    if (st == cudaSuccess) st = cudaMalloc(reinterpret_cast<void**>(&h->t_dirty), (size_t)T);
    if (st == cudaSuccess) st = cudaMalloc(reinterpret_cast<void**>(&h->t_cprev), 2 * sizeof(long long));
    // The tables are written on the handle's stream, ahead of the decisions
    // that read them; the stream is drained before the host tables go away.
    if (st == cudaSuccess) st = cudaMemsetAsync(h->t_dirty, 1, (size_t)T, h->stream);
    if (st == cudaSuccess)
        st = cudaMemsetAsync(h->t_cprev, 0xff, 2 * sizeof(long long), h->stream);   // none yet
    if (st == cudaSuccess)
        st = cudaMemcpyAsync(h->t_items, items.data(), ni * sizeof(fasgd::TensorItem),
                             cudaMemcpyHostToDevice, h->stream);
    if (st == cudaSuccess)
        st = cudaMemcpyAsync(h->t_item_begin, begin.data(), begin.size() * sizeof(int32_t),
                             cudaMemcpyHostToDevice, h->stream);
    if (st == cudaSuccess)
        st = cudaMemcpyAsync(h->t_sizes, sz.data(), sz.size() * sizeof(int32_t),
                             cudaMemcpyHostToDevice, h->stream);
    if (st == cudaSuccess) st = cudaStreamSynchronize(h->stream);
    if (st != cudaSuccess) {
        h->free_tensors();
        return h->cuda_fail(st, "bfasgd_set_tensors");
    }
    h->t_nitems = (int32_t)ni;
    h->tensor_sizes.assign(sizes, sizes + T);
    return FASGD_OK;
}

int bfasgd_push_budget(fasgd_t* h, int32_t client, int64_t timestamp, const float* grad,
                       int64_t budget, uint8_t* sent_dev, float* c_dev, int64_t* count_dev) {
    if (h == nullptr) return FASGD_EINVAL;
    if (h->tensor_sizes.empty()) return h->fail(FASGD_EINVAL, "no tensor partition (bfasgd_set_tensors)");
    if (grad == nullptr || !aligned(grad, 16))
        return h->fail(FASGD_EINVAL, "grad must be a non-NULL 16-byte aligned device pointer");
    if (budget < 0) return h->fail(FASGD_EINVAL, "budget must be >= 0");
    if (!aligned(c_dev, 4) || !aligned(count_dev, 8))
        return h->fail(FASGD_EINVAL, "c_dev must be 4-byte and count_dev 8-byte aligned");
    int rc = check_push(h, client, timestamp);
    if (rc != FASGD_OK) return rc;
    Push p{kBudget, client, timestamp, grad, nullptr, nullptr, nullptr, 0, -1, nullptr,
           budget, sent_dev, c_dev, count_dev};
    h->fifo.push_back(p);
    return FASGD_OK;
}

int bfasgd_fetch_budget(fasgd_t* h, int32_t client, float* theta_client, int64_t budget,
                        uint8_t* sent_dev, float* c_dev, int64_t* count_dev) {
    TraceRange trace("bfasgd_fetch_budget");
    if (h == nullptr) return FASGD_EINVAL;
    if (h->tensor_sizes.empty()) return h->fail(FASGD_EINVAL, "no tensor partition (bfasgd_set_tensors)");
    if (client < 0 || client >= h->lambda)
        return h->fail(FASGD_ERANGE, "client %d outside [0, %d)", client, h->lambda);
    if (theta_client == nullptr || !aligned(theta_client, 16))
        return h->fail(FASGD_EINVAL, "theta_client must be a non-NULL 16-byte aligned device pointer");
    if (budget < 0) return h->fail(FASGD_EINVAL, "budget must be >= 0");
    if (!aligned(c_dev, 4) || !aligned(count_dev, 8))
        return h->fail(FASGD_EINVAL, "c_dev must be 4-byte and count_dev 8-byte aligned");
    DeviceGuard g(h->device);
    cudaError_t st = h->launch_budget(1, client, budget, sent_dev, c_dev, count_dev, h->fetch_count);
    if (st == cudaSuccess) {
        fasgd::RangeArgs r = h->range_args();
        r.src = h->theta;
        r.dst = theta_client;
        st = fasgd::launch_tensor_copy(r, h->stream, &h->launches);
    }
    if (st != cudaSuccess) return h->cuda_fail(st, "bfasgd_fetch_budget");
    return FASGD_OK;
}

int bfasgd_message_vbar(fasgd_t* h, float* vbar_dev) {
    TraceRange trace("bfasgd_message_vbar");
    if (h == nullptr) return FASGD_EINVAL;
    if (vbar_dev == nullptr || !aligned(vbar_dev, 4))
        return h->fail(FASGD_EINVAL, "vbar_dev must be a non-NULL 4-byte aligned device pointer");
    DeviceGuard g(h->device);
    cudaError_t st = h->ensure_message_scratch(false);
    if (st == cudaSuccess)
        st = h->launch_message(0, 0, nullptr, nullptr, nullptr, h->c_push, nullptr, vbar_dev);
    if (st != cudaSuccess) return h->cuda_fail(st, "bfasgd_message_vbar");
    return FASGD_OK;
}

int fasgd_push_sparse(fasgd_t* h, int32_t client, int64_t timestamp, const int32_t* idx,
                      const float* val, const int64_t* n_dev, int64_t n_max) {
    if (h == nullptr) return FASGD_EINVAL;
    if (n_max < 0 || n_max > h->P) return h->fail(FASGD_EINVAL, "n_max must be in [0, P]");
    if (n_max > 0 && (idx == nullptr || val == nullptr))
        return h->fail(FASGD_EINVAL, "idx and val must be non-NULL");
    if (!aligned(idx, 4) || !aligned(val, 4) || !aligned(n_dev, 8))
        return h->fail(FASGD_EINVAL, "idx, val must be 4-byte and n_dev 8-byte aligned");
    int rc = check_push(h, client, timestamp);
    if (rc != FASGD_OK) return rc;
    h->fifo.push_back(Push{kSparse, client, timestamp, nullptr, idx, val, n_dev, n_max, -1, nullptr});
    return FASGD_OK;
}

int fasgd_apply_pending(fasgd_t* h, int32_t K) {
    TraceRange trace("fasgd_apply_pending");
    if (h == nullptr) return FASGD_EINVAL;
    if (K < 1 || K > FASGD_KMAX) return h->fail(FASGD_EINVAL, "K must be in [1, %d]", FASGD_KMAX);
    if ((int64_t)h->fifo.size() < K)
        return h->fail(FASGD_EAGAIN, "K=%d but only %zu pushes pending", K, h->fifo.size());
    DeviceGuard g(h->device);
    const int rule = h->variant == FASGD_FASGD       ? fasgd::kRuleFasgd
                     : h->variant == FASGD_FASGD_STD ? fasgd::kRuleFasgdStd
                                                     : fasgd::kRuleSgd;
    const fasgd::StatParams sp = h->stat_params();
    // Takes the first `done` pushes out of the queue (their passes are
    // enqueued) and advances T past them.  A launch that fails partway keeps
    // the batch's earlier pushes applied: they leave the queue, the failed
    // push and the rest stay, so a retry applies each push exactly once.
    auto retire = [h](int done) {
        for (int i = 0; i < done; ++i) {
            const int slot = h->fifo.front().stage;
            if (slot >= 0) h->stage_busy[(size_t)slot] = 0;
            h->fifo.pop_front();
        }
        h->T += done;
    };
    auto partial_fail = [h, K, &retire](cudaError_t st, const char* what, int done) {
        retire(done);
        return h->fail(st == cudaErrorMemoryAllocation ? FASGD_ENOMEM : FASGD_ECUDA,
                       "fasgd_apply_pending: %s: %s (%d of %d pushes were applied and left the "
                       "queue; T advanced by %d)", what, cudaGetErrorString(st), done, K, done);
    };
    int k = 0;
    while (k < K) {
        const Push& first = h->fifo[(size_t)k];
        if (first.kind != kBudget) h->t_sums_valid = false;   // this pass rewrites v
        if (first.kind != kMessage) h->msg_sums_valid = false;
        if (first.kind == kDense) {
            // Fuse the run of consecutive dense pushes into one pass.
            fasgd::DenseArgs a;
            std::memset(&a, 0, sizeof a);
            a.theta = h->theta;
            a.n = h->n;
            a.b = h->b;
            a.v = h->v;
            a.P = h->P;
            a.sp = sp;
            a.err = h->dev_err;
            int r = 0;
            while (k + r < K && h->fifo[(size_t)(k + r)].kind == kDense) {
                const Push& p = h->fifo[(size_t)(k + r)];
                a.grad[r] = p.grad;
                a.coef[r] = h->coef(h->T + k + r - p.j);
                ++r;
            }
            a.K = r;
            cudaError_t st = cudaSuccess;
            for (int i = 0; i < r && st == cudaSuccess; ++i) {  // staged host copies landed
                const int slot = h->fifo[(size_t)(k + i)].stage;
                if (slot >= 0) st = cudaStreamWaitEvent(h->stream, h->slot_ready[(size_t)slot], 0);
            }
            if (st == cudaSuccess)
                st = h->injected_failure()
                         ? cudaErrorLaunchFailure
                         : fasgd::launch_dense(a, rule, h->exact, h->num_sms, h->stream, &h->launches);
            ++h->pass_seq;
            for (int i = 0; i < r && st == cudaSuccess; ++i) {  // the slots may be refilled after this
                const int slot = h->fifo[(size_t)(k + i)].stage;
                if (slot >= 0) {
                    st = cudaEventRecord(h->slot_free[(size_t)slot], h->stream);
                    h->stage_used[(size_t)slot] = 1;
                    h->stage_seq[(size_t)slot] = h->pass_seq;
                }
            }
            if (st != cudaSuccess) return partial_fail(st, "dense pass", k);
            k += r;
        } else if (first.kind == kMessage) {
            // Decide against the mean of v now, refresh the client's cache
            // slot if the push is transmitted, then apply the slot.  Under the
            // FASGD rules the pass itself takes the decision from the
            // statistic's partials and, if transmitted, applies the pushed
            // gradient while copying it into the slot.
            float* slot = h->grad_cache + (size_t)first.client * (size_t)h->cache_stride;
            const uint64_t count0 = h->push_count[(size_t)first.client];
            fasgd::DenseArgs a;
            std::memset(&a, 0, sizeof a);
            a.theta = h->theta;
            a.n = h->n;
            a.b = h->b;
            a.v = h->v;
            a.P = h->P;
            a.sp = sp;
            a.err = h->dev_err;
            a.grad[0] = slot;
            a.coef[0] = h->coef(h->T + k - first.j);
            a.K = 1;
            cudaError_t st;
            if (rule != fasgd::kRuleSgd) {
                const fasgd::MessageArgs m =
                    h->message_args(0, first.client, first.grad, slot, first.flag, h->c_push,
                                    count0, nullptr);
                st = fasgd::launch_message_partials(m, h->stream, &h->launches);
                if (st == cudaSuccess) {
                    a.vsum = h->msg_chunks;   // keep the chunk sums current
                    a.msg.partial = m.partial;
                    a.msg.nblocks = m.nblocks;
                    a.msg.c = m.c;
                    a.msg.eps_b = m.eps_b;
                    std::memcpy(a.msg.round_key0, m.round_key0, sizeof a.msg.round_key0);
                    std::memcpy(a.msg.round_key1, m.round_key1, sizeof a.msg.round_key1);
                    a.msg.client_word = m.client_word;
                    a.msg.n_lo = m.n_lo;
                    a.msg.n_hi = m.n_hi;
                    a.msg.src = first.grad;
                    a.msg.slot = slot;
                    a.msg.flag_out = first.flag;
                    st = h->injected_failure()
                             ? cudaErrorLaunchFailure
                             : fasgd::launch_dense(a, rule, h->exact, h->num_sms, h->stream,
                                                   &h->launches);
                    if (st == cudaSuccess) h->push_count[(size_t)first.client] = count0 + 1;
                }
                h->msg_sums_valid = st == cudaSuccess;
            } else {
                st = h->launch_message(0, first.client, first.grad, slot, first.flag, h->c_push,
                                       &h->push_count);
                if (st == cudaSuccess)
                    st = h->injected_failure()
                             ? cudaErrorLaunchFailure
                             : fasgd::launch_dense(a, rule, h->exact, h->num_sms, h->stream,
                                                   &h->launches);
                h->msg_sums_valid = st == cudaSuccess;
            }
            if (st != cudaSuccess) {
                // A retry redraws the same decision against the same v (the
                // pass did not run), so it refreshes the cache slot alike.
                h->push_count[(size_t)first.client] = count0;
                return partial_fail(st, "message push", k);
            }
            k += 1;
        } else if (first.kind == kBudget) {
            // Decide every tensor against the statistics now, then update the
            // transmitted ones.
            const uint64_t count0 = h->push_count[(size_t)first.client];
            cudaError_t st = h->launch_budget(0, first.client, first.budget, first.sent_out,
                                              first.c_out, first.count_out, h->push_count);
            if (st == cudaSuccess) {
                fasgd::RangeArgs r = h->range_args();
                r.grad = first.grad;
                r.coef = h->coef(h->T + k - first.j);
                st = h->injected_failure()
                         ? cudaErrorLaunchFailure
                         : fasgd::launch_tensor_apply(r, rule, h->exact, h->stream, &h->launches);
            }
            if (st != cudaSuccess) {
                h->push_count[(size_t)first.client] = count0;   // a retry redraws the same decision
                return partial_fail(st, "budget push", k);
            }
            k += 1;
        } else {
            fasgd::SparseArgs a;
            std::memset(&a, 0, sizeof a);
            a.theta = h->theta;
            a.n = h->n;
            a.b = h->b;
            a.v = h->v;
            a.idx = first.idx;
            a.val = first.val;
            a.count_dev = first.n_dev;
            a.count_max = first.n_max;
            a.P = h->P;
            a.coef = h->coef(h->T + k - first.j);
            a.sp = sp;
            a.err = h->dev_err;
            if (first.n_max > 0 || first.n_dev != nullptr) {
                cudaError_t st = h->injected_failure()
                                     ? cudaErrorLaunchFailure
                                     : fasgd::launch_sparse(a, rule, h->exact, h->num_sms, h->stream,
                                                            &h->launches);
                if (st != cudaSuccess) return partial_fail(st, "sparse pass", k);
            }
            k += 1;
        }
    }
    retire(K);
    return FASGD_OK;
}

}  // extern "C"

// One B-FASGD decision + compaction pass: stream 0 (push: values = the
// client's gradient, threshold c_push) or 1 (fetch: values = theta, c_fetch).
static int run_select(fasgd_t* h, const char* what, uint32_t stream, int32_t client,
                      const float* values, const float* v, int32_t* idx, float* val,
                      int64_t* n_dev, float c, std::vector<uint64_t>& counter) {
    TraceRange trace(what);
    if (client < 0 || client >= h->lambda)
        return h->fail(FASGD_ERANGE, "%s: client %d outside [0, %d)", what, client, h->lambda);
    if (values == nullptr || !aligned(values, 16))
        return h->fail(FASGD_EINVAL, "%s: grad must be a non-NULL 16-byte aligned device pointer",
                       what);
    if (v != nullptr && !aligned(v, 16))
        return h->fail(FASGD_EINVAL, "%s: v must be 16-byte aligned (or NULL for the server's v)",
                       what);
    if (idx == nullptr || val == nullptr || n_dev == nullptr || !aligned(idx, 4) ||
        !aligned(val, 4) || !aligned(n_dev, 8))
        return h->fail(FASGD_EINVAL, "%s: idx, val, n_dev must be non-NULL and aligned", what);
    DeviceGuard g(h->device);
    fasgd::SelectArgs a;
    std::memset(&a, 0, sizeof a);
    a.values = values;
    a.v = v != nullptr ? v : h->v;
    a.idx = idx;
    a.val = val;
    a.count = n_dev;
    a.mask = h->mask;
    a.tile_count = h->tile_count;
    a.tile_base = h->tile_base;
    a.P = h->P;
    a.ntiles = h->ntiles;
    a.c = c;
    a.eps_b = h->eps_b;
    fasgd::select_key_schedule(a, h->seed);
    const uint64_t n = counter[(size_t)client];
    a.client_word = (uint32_t)client | (stream << 31);
    a.push_lo = (uint32_t)n;
    a.push_hi = (uint32_t)(n >> 32);
    cudaError_t st = fasgd::launch_select(a, h->stream, &h->launches);
    if (st != cudaSuccess) return h->cuda_fail(st, what);
    counter[(size_t)client] = n + 1;
    return FASGD_OK;
}

extern "C" {

int bfasgd_select_compact(fasgd_t* h, int32_t client, const float* grad, const float* v,
                          int32_t* idx, float* val, int64_t* n_dev) {
    if (h == nullptr) return FASGD_EINVAL;
    return run_select(h, "bfasgd_select_compact", 0, client, grad, v, idx, val, n_dev, h->c_push,
                      h->push_count);
}

int bfasgd_fetch_compact(fasgd_t* h, int32_t client, const float* v, int32_t* idx, float* val,
                         int64_t* n_dev) {
    if (h == nullptr) return FASGD_EINVAL;
    return run_select(h, "bfasgd_fetch_compact", 1, client, h->theta, v, idx, val, n_dev,
                      h->c_fetch, h->fetch_count);
}

int fasgd_set_fetch_threshold(fasgd_t* h, float c_fetch) {
    if (h == nullptr) return FASGD_EINVAL;
    if (!(c_fetch >= 0.f)) return h->fail(FASGD_EINVAL, "c_fetch must be >= 0 (may be +inf)");
    h->c_fetch = c_fetch;
    return FASGD_OK;
}

int bfasgd_fetch_apply(int64_t P, float* theta_client, const int32_t* idx, const float* val,
                       const int64_t* n_dev, int64_t n_max, void* stream, int32_t* err_dev) {
    TraceRange trace("bfasgd_fetch_apply");
    if (P < 1 || P > FASGD_PMAX) {
        g_create_error = "bfasgd_fetch_apply: P must be in [1, 2^31)";
        return FASGD_EINVAL;
    }
    if (theta_client == nullptr || n_max < 0 || n_max > P ||
        (n_max > 0 && (idx == nullptr || val == nullptr)) || !aligned(theta_client, 4) ||
        !aligned(idx, 4) || !aligned(val, 4) || !aligned(n_dev, 8) || !aligned(err_dev, 4)) {
        g_create_error = "bfasgd_fetch_apply: bad pointer or n_max outside [0, P]";
        return FASGD_EINVAL;
    }
    if (n_max == 0 && n_dev == nullptr) return FASGD_OK;
    int dev = 0, sms = 0;
    cudaError_t st = cudaGetDevice(&dev);
    if (st == cudaSuccess) st = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    fasgd::ScatterArgs a;
    a.theta = theta_client;
    a.idx = idx;
    a.val = val;
    a.count_dev = n_dev;
    a.count_max = n_max;
    a.P = P;
    a.err = err_dev;
    if (st == cudaSuccess) st = fasgd::launch_scatter(a, sms, static_cast<cudaStream_t>(stream));
    if (st != cudaSuccess) {
        g_create_error = std::string("bfasgd_fetch_apply: ") + cudaGetErrorString(st);
        return FASGD_ECUDA;
    }
    return FASGD_OK;
}

int fasgd_sim_quadratic_grad(int64_t P, const float* theta, const float* hcurv, const float* star,
                             const float* sigma, uint64_t seed, int32_t client, uint64_t n,
                             float* grad, void* stream) {
    if (P < 1 || P > FASGD_PMAX || client < 0 || client >= (1 << 30)) {
        g_create_error = "fasgd_sim_quadratic_grad: P or client out of range";
        return FASGD_EINVAL;
    }
    const void* ptrs[] = {theta, hcurv, star, sigma, grad};
    for (const void* q : ptrs)
        if (q == nullptr || !aligned(q, 16)) {
            g_create_error = "fasgd_sim_quadratic_grad: pointers must be non-NULL, 16-byte aligned";
            return FASGD_EINVAL;
        }
    int dev = 0, sms = 0;
    cudaError_t st = cudaGetDevice(&dev);
    if (st == cudaSuccess) st = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    fasgd::SimGradArgs a;
    a.theta = theta;
    a.h = hcurv;
    a.star = star;
    a.sigma = sigma;
    a.grad = grad;
    a.P = P;
    fasgd::philox_key_schedule(seed, a.round_key0, a.round_key1);
    a.client = (uint32_t)client;
    a.n_lo = (uint32_t)n;
    a.n_hi = (uint32_t)(n >> 32);
    if (st == cudaSuccess) st = fasgd::launch_sim_grad(a, sms, static_cast<cudaStream_t>(stream));
    if (st != cudaSuccess) {
        g_create_error = std::string("fasgd_sim_quadratic_grad: ") + cudaGetErrorString(st);
        return FASGD_ECUDA;
    }
    return FASGD_OK;
}

int fasgd_sim_quadratic_loss(int64_t P, const float* theta, const float* hcurv, const float* star,
                             double* scratch, double* loss, void* stream) {
    if (P < 1 || P > FASGD_PMAX || theta == nullptr || hcurv == nullptr || star == nullptr ||
        scratch == nullptr || loss == nullptr || !aligned(scratch, 8) || !aligned(loss, 8)) {
        g_create_error = "fasgd_sim_quadratic_loss: bad argument";
        return FASGD_EINVAL;
    }
    fasgd::SimLossArgs a;
    a.theta = theta;
    a.h = hcurv;
    a.star = star;
    a.P = P;
    a.partial = scratch;
    a.loss = loss;
    cudaError_t st = fasgd::launch_sim_loss(a, static_cast<cudaStream_t>(stream));
    if (st != cudaSuccess) {
        g_create_error = std::string("fasgd_sim_quadratic_loss: ") + cudaGetErrorString(st);
        return FASGD_ECUDA;
    }
    return FASGD_OK;
}

int fasgd_pull(fasgd_t* h, float* params, int64_t* T) {
    TraceRange trace("fasgd_pull");
    if (h == nullptr) return FASGD_EINVAL;
    if (params != nullptr) {
        // The copy runs on its own stream (so it overlaps host-push copies of
        // the next pushes) and the handle's stream waits for it: later work on
        // the stream, and a caller synchronising it, see the pull complete.
        DeviceGuard g(h->device);
        cudaError_t st = h->ensure_aux();
        if (st == cudaSuccess) st = cudaEventRecord(h->order_ev, h->stream);
        if (st == cudaSuccess) st = cudaStreamWaitEvent(h->pull_stream, h->order_ev, 0);
        if (st == cudaSuccess)
            st = cudaMemcpyAsync(params, h->theta, (size_t)h->P * sizeof(float), cudaMemcpyDefault,
                                 h->pull_stream);
        if (st == cudaSuccess) st = cudaEventRecord(h->pull_done_ev, h->pull_stream);
        if (st == cudaSuccess) st = cudaStreamWaitEvent(h->stream, h->pull_done_ev, 0);
        if (st != cudaSuccess) return h->cuda_fail(st, "fasgd_pull");
    }
    if (T != nullptr) *T = h->T;
    return FASGD_OK;
}

int fasgd_get_state(fasgd_t* h, float* theta, float* n, float* b, float* v, int64_t* T) {
    TraceRange trace("fasgd_get_state");
    if (h == nullptr) return FASGD_EINVAL;
    if (!h->fifo.empty()) return h->fail(FASGD_EAGAIN, "pushes are pending");
    DeviceGuard g(h->device);
    float* dst[] = {theta, n, b, v};
    const float* src[] = {h->theta, h->n, h->b, h->v};
    for (int i = 0; i < 4; ++i) {
        if (dst[i] == nullptr) continue;
        cudaError_t st = cudaMemcpyAsync(dst[i], src[i], (size_t)h->P * sizeof(float),
                                         cudaMemcpyDefault, h->stream);
        if (st != cudaSuccess) return h->cuda_fail(st, "fasgd_get_state");
    }
    cudaError_t st = cudaStreamSynchronize(h->stream);
    if (st != cudaSuccess) return h->cuda_fail(st, "fasgd_get_state");
    if (T != nullptr) *T = h->T;
    return FASGD_OK;
}

int fasgd_set_state(fasgd_t* h, const float* theta, const float* n, const float* b,
                    const float* v, int64_t T) {
    TraceRange trace("fasgd_set_state");
    if (h == nullptr) return FASGD_EINVAL;
    if (T < 0) return h->fail(FASGD_EINVAL, "T must be >= 0");
    if (!h->fifo.empty()) return h->fail(FASGD_EAGAIN, "pushes are pending");
    DeviceGuard g(h->device);
    float* dst[] = {h->theta, h->n, h->b, h->v};
    const float* src[] = {theta, n, b, v};
    for (int i = 0; i < 4; ++i) {
        if (src[i] == nullptr) continue;
        cudaError_t st = cudaMemcpyAsync(dst[i], src[i], (size_t)h->P * sizeof(float),
                                         cudaMemcpyDefault, h->stream);
        if (st != cudaSuccess) return h->cuda_fail(st, "fasgd_set_state");
    }
    h->T = T;
    if (v != nullptr) {
        h->t_sums_valid = false;
        h->msg_sums_valid = false;
    }
    return FASGD_OK;
}

int fasgd_get_push_counts(fasgd_t* h, uint64_t* counts) {
    if (h == nullptr || counts == nullptr) return FASGD_EINVAL;
    std::memcpy(counts, h->push_count.data(), h->push_count.size() * sizeof(uint64_t));
    return FASGD_OK;
}

int fasgd_set_push_counts(fasgd_t* h, const uint64_t* counts) {
    if (h == nullptr || counts == nullptr) return FASGD_EINVAL;
    std::memcpy(h->push_count.data(), counts, h->push_count.size() * sizeof(uint64_t));
    return FASGD_OK;
}

int fasgd_get_fetch_counts(fasgd_t* h, uint64_t* counts) {
    if (h == nullptr || counts == nullptr) return FASGD_EINVAL;
    std::memcpy(counts, h->fetch_count.data(), h->fetch_count.size() * sizeof(uint64_t));
    return FASGD_OK;
}

int fasgd_set_fetch_counts(fasgd_t* h, const uint64_t* counts) {
    if (h == nullptr || counts == nullptr) return FASGD_EINVAL;
    std::memcpy(h->fetch_count.data(), counts, h->fetch_count.size() * sizeof(uint64_t));
    return FASGD_OK;
}

int fasgd_sync(fasgd_t* h) {
    if (h == nullptr) return FASGD_EINVAL;
    DeviceGuard g(h->device);
    cudaError_t st = cudaStreamSynchronize(h->stream);
    if (st != cudaSuccess) return h->cuda_fail(st, "fasgd_sync");
    int32_t flags = 0;
    st = cudaMemcpy(&flags, h->dev_err, sizeof flags, cudaMemcpyDeviceToHost);
    if (st != cudaSuccess) return h->cuda_fail(st, "fasgd_sync");
    if (flags != 0) {
        st = cudaMemset(h->dev_err, 0, sizeof(int32_t));
        if (st == cudaSuccess) st = cudaDeviceSynchronize();
        if (st != cudaSuccess) return h->cuda_fail(st, "fasgd_sync");
        return h->fail(FASGD_EDEVICE, "device error flags 0x%x (1: sparse count > n_max, "
                                      "2: sparse index out of range, 4: sparse indices not "
                                      "ascending, 8: a dense-pass pipeline wait expired)", flags);
    }
    return FASGD_OK;
}

int fasgd_selftest_wait_expiry(fasgd_t* h) {
    if (h == nullptr) return FASGD_EINVAL;
    TraceRange trace("fasgd_selftest_wait_expiry");
    DeviceGuard g(h->device);
    cudaError_t st = fasgd::launch_wait_expiry(h->dev_err, h->stream);
    if (st != cudaSuccess) return h->cuda_fail(st, "fasgd_selftest_wait_expiry");
    ++h->launches;
    return FASGD_OK;
}

int fasgd_selftest_fail_pass(fasgd_t* h, int32_t after) {
    if (h == nullptr) return FASGD_EINVAL;
    if (after < -1) return h->fail(FASGD_EINVAL, "after must be >= -1");
    h->fail_pass_in = after;
    return FASGD_OK;
}

int64_t fasgd_timestamp(const fasgd_t* h) { return h == nullptr ? -1 : h->T; }

int64_t fasgd_pending(const fasgd_t* h) { return h == nullptr ? -1 : (int64_t)h->fifo.size(); }

int64_t fasgd_kernel_launches(const fasgd_t* h) { return h == nullptr ? -1 : h->launches; }

const char* fasgd_last_error(const fasgd_t* h) {
    return h == nullptr ? g_create_error.c_str() : h->err.c_str();
}

}  // extern "C"
