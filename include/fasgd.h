/*
 * fasgd.h -- C ABI of the GB300 FASGD parameter-server library.
 *
 * The library is the server side of "Faster Asynchronous SGD" (Odena, 2016):
 * it keeps the parameter vector theta and the per-parameter gradient
 * statistics n, b, v in device memory, queues client pushes in arrival
 * order, and applies them with the update rules of Sec. 2.1-2.2
 * (ASGD, SASGD Eq. 1-2, FASGD Eq. 4-8).  It also implements the push side
 * of B-FASGD (Sec. 2.3, Eq. 9) per parameter: the send decision, the
 * compaction of the sent entries into index/value lists, and the sparse
 * server apply of such lists.
 *
 * Conventions shared by every call
 *   - Return value: FASGD_OK (0) or a negative fasgd_status.  A call that
 *     fails validation changes no state.  fasgd_last_error() describes the
 *     most recent failure on a handle (or, with NULL, of fasgd_create).
 *   - Asynchrony: every call that touches device memory is enqueued on the
 *     handle's stream (fasgd_set_stream) and returns before the GPU is done.
 *     Only values written to host memory by the call itself (timestamps,
 *     counts) are final on return.  Device-side checks on caller-supplied
 *     index lists are reported by fasgd_sync().
 *   - Ownership: the handle owns theta, n, b, v and its scratch buffers.
 *     Every other pointer belongs to the caller and is only borrowed; a
 *     buffer passed to fasgd_push / fasgd_push_sparse must stay valid and
 *     unmodified until the fasgd_apply_pending call that consumes it has
 *     completed on the stream.
 *   - Pointers: "device" pointers must be device-accessible (cudaMalloc,
 *     torch CUDA tensors).  Dense fp32[P] vectors (gradients, v) must be
 *     16-byte aligned (they are read 128 bits at a time); index / value
 *     lists 4-byte and counts 8-byte aligned.  "host or device" pointers may
 *     also be host memory (pinned host memory keeps the copy asynchronous).
 *   - Sizes: 1 <= P < 2^31 (indices are int32), 1 <= lambda <= 2^20,
 *     1 <= K <= FASGD_KMAX pushes per apply.
 *   - Threads: a handle is used by one host thread at a time.
 */
#ifndef FASGD_H
#define FASGD_H

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef struct fasgd_s fasgd_t;

/* Every entry point is exported from the shared library. */
#if defined(__GNUC__)
#define FASGD_API __attribute__((visibility("default")))
#else
#define FASGD_API
#endif

/* Update rule of the server (Sec. 2.1-2.2). */
enum fasgd_variant {
    FASGD_ASGD = 0,   /* theta -= alpha * g                       (Sec. 2.1, protocol step 2) */
    FASGD_SASGD = 1,  /* theta -= alpha / max(tau,1) * g           (Eq. 1-2) */
    FASGD_FASGD = 2,  /* n, b, v moving averages, then
                         theta -= alpha / (v * max(tau,1)) * g     (Eq. 4-8) */
    FASGD_FASGD_STD = 3  /* as FASGD, but v averages the std sqrt(n - b^2 + eps)
                            itself, so the step is divided by the std: the
                            reading of Sec. 2.2's prose ("dividing the learning
                            rate by the standard deviation") */
};

enum fasgd_status {
    FASGD_OK = 0,
    FASGD_EINVAL = -1,   /* bad argument: NULL or misaligned pointer, size or
                            hyper-parameter outside its domain, bad variant */
    FASGD_ERANGE = -2,   /* client outside [0, lambda) or timestamp outside [0, T] */
    FASGD_EAGAIN = -3,   /* fewer than K pending pushes, queue or staging full,
                            or pushes still pending where none may be */
    FASGD_ENOMEM = -4,   /* device or pinned allocation failed */
    FASGD_ECUDA = -5,    /* a CUDA runtime call failed (text in fasgd_last_error) */
    FASGD_EDEVICE = -6   /* a kernel found a bad entry in a caller's sparse list */
};

#define FASGD_KMAX 32                         /* pushes one apply may fuse */
#define FASGD_PMAX ((int64_t)2147483647)      /* P must be below 2^31 */

/*
 * fasgd_create -- make a server with P fp32 parameters for lambda clients.
 * Sec. 2.1 notation: lambda clients, master learning rate alpha, timestamp
 * T starting at 0.  theta, n, b, v are allocated on the current CUDA device
 * and zero-filled (the statistics start at 0; set theta with
 * fasgd_set_params).  Default hyper-parameters: gamma = beta = 0.95,
 * eps = 1e-4, c_push = 0 (send everything), eps_b = 1e-8, seed = 0.
 * Errors: EINVAL (h NULL, P or lambda out of range, alpha not finite, bad
 * variant), ENOMEM, ECUDA.  On error *h is set to NULL.
 */
FASGD_API int fasgd_create(fasgd_t** h, int64_t P, int32_t lambda, float alpha, int32_t variant);

/* Free every device buffer of the handle (after the stream drains).  NULL is ignored. */
FASGD_API void fasgd_destroy(fasgd_t* h);

/*
 * fasgd_set_hparams -- gamma, beta (Eq. 4-6 moving-average factors),
 * eps (Eq. 6 stabiliser), c_push and eps_b (Eq. 9 threshold and its
 * stabiliser) and the 64-bit seed of the B-FASGD draws.
 * Domain: 0 <= gamma <= 1, 0 <= beta < 1, eps and eps_b finite and >= 0,
 * c_push >= 0 (+inf allowed: nothing is sent).  The send decision is exact
 * for every v_p >= 0 of any finite magnitude (subnormal to FLT_MAX) and
 * every c_push >= 0; a parameter with v_p + eps_b = 0 is never sent, and
 * (v_p + eps_b) + c_push must stay below 2^128 unless c_push = +inf (a
 * finite sum that rounds to +inf in fp32 would read as "never sent").
 * Errors: EINVAL (outside the domain), EAGAIN (pushes pending).
 */
FASGD_API int fasgd_set_hparams(fasgd_t* h, float gamma, float beta, float eps, float c_push,
                      float eps_b, uint64_t seed);

/*
 * fasgd_set_exact -- choose the arithmetic of the FASGD update (Eq. 4-8):
 * 0 (default) uses the hardware inverse square root / reciprocal and fused
 * multiply-adds for v and theta; 1 computes every operation correctly
 * rounded and unfused -- the exact fp32 sequence, bit for bit what an IEEE
 * CPU computes.  n and b are exact in both modes, and so are ASGD/SASGD.
 *
 * Where mode 0 holds 1e-5 relative: v is a weighted mean, so its error stays
 * at a few ulp; theta's error is a few ulp of the largest |theta| the
 * parameter passes through, since each step carries a few ulp of error
 * relative to its own size.  So theta stays within 1e-5 * |theta| + 1e-7 of
 * the exact sequence while no parameter swings far above where it ends --
 * roughly while max |theta| along the run stays below 25 |theta_end| or
 * below 0.3.  Steps of order |theta| break that: the divide-by-std rule at
 * FASGD's learning rates, or beta near 1 (the first v is (1 - beta) r, so
 * the first steps are large).  Measured: theta through 3.2 ending at 5.6e-3
 * is 7e-7 off (1.14 times the bound).  Use mode 1 there, and wherever runs
 * must reproduce exactly (closed-loop simulations, where feedback can
 * amplify ulp-level differences).  Mode 1 costs about 1.9x per dense pass
 * at K = 8.  Errors: EINVAL, EAGAIN (pushes pending).
 */
FASGD_API int fasgd_set_exact(fasgd_t* h, int32_t exact);

/*
 * Stream every later call is enqueued on (a cudaStream_t; NULL = legacy
 * default stream).  Work the handle already enqueued on the previous stream
 * comes before anything it enqueues on the new one: the call records an event
 * on the previous stream and makes the new stream wait for it (so neither
 * stream may be in a stream capture that the other is not part of).
 * Errors: EINVAL, EAGAIN (pushes pending), ECUDA (the event could not be
 * recorded or waited on; the stream is not changed).
 */
FASGD_API int fasgd_set_stream(fasgd_t* h, void* stream);

/*
 * fasgd_set_params -- copy P initial parameters (host or device pointer)
 * into theta.  n, b, v are left as they are.  Errors: EINVAL, EAGAIN
 * (pushes pending), ECUDA.
 */
FASGD_API int fasgd_set_params(fasgd_t* h, const float* theta0);

/*
 * fasgd_push -- queue one dense client gradient (Sec. 2.1, protocol step 1).
 * client in [0, lambda); timestamp j = the server timestamp of the
 * parameters the gradient was computed on, 0 <= j <= T (T = the server's
 * current timestamp; pushes already queued do not advance it).
 * grad: device pointer to P fp32 values, 16-byte aligned, borrowed until
 * the apply that consumes it completes on the stream.
 * Errors: EINVAL, ERANGE, EAGAIN (queue holds 2^20 pushes).
 */
FASGD_API int fasgd_push(fasgd_t* h, int32_t client, int64_t timestamp, const float* grad);

/*
 * fasgd_push_host -- as fasgd_push, for a gradient in host memory: the P
 * values are copied asynchronously into a device staging slot owned by the
 * handle, on an internal copy stream so that the copies of later pushes
 * overlap the pass that consumes earlier ones (the pass waits for its
 * copies).  The host buffer must stay unchanged until the apply that
 * consumes the push has completed on the handle's stream (pinned memory
 * keeps the copy asynchronous).  At most FASGD_KMAX host pushes may be
 * pending; staging slots (P floats each, at most FASGD_KMAX) are allocated on
 * first need.  Errors: EINVAL, ERANGE, EAGAIN, ENOMEM, ECUDA.
 */
FASGD_API int fasgd_push_host(fasgd_t* h, int32_t client, int64_t timestamp, const float* grad_host);

/*
 * fasgd_push_sparse -- queue one sparse push: parameter idx[i] receives
 * gradient entry val[i] for i < count; every other parameter is left alone
 * (its statistics do not decay).  This is the server side of a B-FASGD push
 * whose unsent entries are dropped.
 * idx: device int32 list, strictly ascending, each in [0, P).
 * val: device fp32 list.  count: read on the device from *n_dev when n_dev
 * is not NULL (as written by bfasgd_select_compact), else count = n_max.
 * n_max: host-side upper bound, 0 <= n_max <= P; idx and val hold at least
 * n_max entries.  All three buffers are borrowed until the consuming apply
 * completes.  A count above n_max, an index out of range or out of order
 * is skipped on the device and reported by fasgd_sync() as EDEVICE.
 * Errors: EINVAL, ERANGE, EAGAIN.
 */
FASGD_API int fasgd_push_sparse(fasgd_t* h, int32_t client, int64_t timestamp, const int32_t* idx,
                      const float* val, const int64_t* n_dev, int64_t n_max);

/*
 * fasgd_apply_pending -- apply the first K queued pushes in arrival order
 * (Sec. 2.1 protocol step 2; Eq. 1-2 or Eq. 4-8 per the variant).  Push k of
 * the batch (k = 0..K-1) is applied at server timestamp T + k, so its
 * step-staleness is tau_k = T + k - j_k, and alpha(tau) = alpha / max(tau,1).
 * Consecutive dense pushes are fused into one pass over the parameters that
 * keeps each element's theta, n, b, v in registers across them; each sparse
 * push is its own pass.  T increases by K.
 * Errors: EINVAL (K < 1 or K > FASGD_KMAX), EAGAIN (fewer than K pending), ECUDA.
 * If a launch fails partway through the batch (ECUDA or ENOMEM), the pushes
 * whose passes were already enqueued count as applied: they have left the
 * queue and T has advanced by their number (the message says how many);
 * the push that failed and the rest of the batch are still queued, with
 * their draw counters unchanged, so retrying applies each push once.
 */
FASGD_API int fasgd_apply_pending(fasgd_t* h, int32_t K);

/*
 * bfasgd_select_compact -- B-FASGD push decision and compaction (Sec. 2.3,
 * Eq. 9, taken per parameter with the parameter's own v_p).
 * For every p, u_p is the top 24 bits of word (p mod 4) of Philox4x32-10
 * (Salmon et al., SC'11) with counter (p div 4, client, push#, push# >> 32)
 * and key = seed, where push# counts this client's earlier pushes.  With
 * a = fl(v_p + eps_b) and d = fl(a + c_push), p is sent iff
 * u_p * d < a * 2^24 exactly, i.e. u_p / 2^24 < 1 / (1 + c_push / a).
 * Outputs: idx[0..m) = the sent p in ascending order (int32), val[i] =
 * grad[idx[i]] (bit copy), *n_dev = m (int64), all written on the stream.
 * grad: device fp32[P]; v: device fp32[P] (the client's copy of the server
 * statistic), or NULL to use the server's live v.  idx, val: device, room
 * for P entries.  Uses handle-owned scratch (a bit mask and per-tile counts).
 * Errors: EINVAL, ERANGE (client), ECUDA.  On success the client's push#
 * advances by one.
 */
FASGD_API int bfasgd_select_compact(fasgd_t* h, int32_t client, const float* grad, const float* v,
                          int32_t* idx, float* val, int64_t* n_dev);

/*
 * bfasgd_fetch_compact -- B-FASGD fetch decision and compaction, per
 * parameter (Sec. 2.3: at each chance to receive fresh parameters a client
 * takes them iff Eq. 9 holds; here with each parameter's own v_p, as the
 * future-work section proposes).  Exactly as
 * bfasgd_select_compact, with the fetch threshold c_fetch
 * (fasgd_set_fetch_threshold), draws from the fetch stream (counter word
 * client + 2^31, push# replaced by the client's count of earlier fetches),
 * and the server's current theta as the values: idx[0..m) = the kept p
 * ascending, val[i] = theta[idx[i]], *n_dev = m.  theta is read as of the
 * pushes applied so far on the stream.  v: device fp32[P] or NULL for the
 * server's live v.  The client applies the result with bfasgd_fetch_apply
 * and keeps its stale values elsewhere.  Errors: EINVAL, ERANGE, ECUDA.
 */
FASGD_API int bfasgd_fetch_compact(fasgd_t* h, int32_t client, const float* v, int32_t* idx,
                                   float* val, int64_t* n_dev);

/* Fetch threshold c_fetch of Eq. 9 (>= 0, +inf allowed: nothing is fetched).  Default 0. */
FASGD_API int fasgd_set_fetch_threshold(fasgd_t* h, float c_fetch);

/*
 * bfasgd_fetch_apply -- client side of a fetch: theta_client[idx[i]] = val[i]
 * for i < count, on `stream` (a cudaStream_t; NULL = legacy default stream).
 * theta_client: device fp32[P]; idx, val: device lists from
 * bfasgd_fetch_compact (distinct indices); count = *n_dev if n_dev is not
 * NULL, else n_max; 0 <= n_max <= P.  An index outside [0, P) is skipped and
 * a count above n_max is clamped; both raise flags in *err_dev (device int32,
 * may be NULL).  Needs no handle.  Errors: EINVAL (text via
 * fasgd_last_error(NULL)), ECUDA.
 */
FASGD_API int bfasgd_fetch_apply(int64_t P, float* theta_client, const int32_t* idx,
                                 const float* val, const int64_t* n_dev, int64_t n_max,
                                 void* stream, int32_t* err_dev);

/*
 * bfasgd_push_message -- the paper's literal B-FASGD push (Sec. 2.3): one
 * decision for the whole message.  When the push is applied (in arrival
 * order, by fasgd_apply_pending), the server forms vbar = the mean of v over
 * all P parameters (a compensated sum in a fixed order, rounded once to fp32), draws u
 * (Philox4x32-10 word 0 at counter (2^32-1, client, n, n >> 32), key = seed,
 * n = the client's push count, which then advances) and transmits iff Eq. 9
 * holds: u / 2^24 < 1 / (1 + c_push / (vbar + eps_b)), decided exactly in
 * fp32.  A transmitted push replaces the client's slot of the server's
 * gradient cache; either way the server applies the slot, so a dropped push
 * re-applies the client's most recent transmitted gradient (zeros if it has
 * none yet) -- the paper's choice.  The first call allocates the cache:
 * lambda x P floats.  grad: device fp32[P], 16-byte aligned, borrowed until
 * the apply completes.  sent_dev: device int32 receiving 1 (transmitted) or 0
 * (dropped) when the push is applied, or NULL.  Such a push is applied as its
 * own pass (it does not fuse with neighbours).
 * Errors: EINVAL, ERANGE, EAGAIN, ENOMEM, ECUDA.
 */
FASGD_API int bfasgd_push_message(fasgd_t* h, int32_t client, int64_t timestamp,
                                  const float* grad, int32_t* sent_dev);

/*
 * bfasgd_fetch_message -- the paper's literal B-FASGD fetch (Sec. 2.3): one
 * decision, as for a message push but with c_fetch and counter word
 * client + 2^31 (n = the client's fetch count, which advances), taken on the
 * stream against the current server state; if transmitted, theta is copied
 * into theta_client (device fp32[P], 16-byte aligned), otherwise the client
 * keeps its copy.  fetched_dev: device int32 receiving 1 or 0, or NULL.
 * Errors: EINVAL, ERANGE, ENOMEM, ECUDA.
 */
FASGD_API int bfasgd_fetch_message(fasgd_t* h, int32_t client, float* theta_client,
                                   int32_t* fetched_dev);

/*
 * bfasgd_message_vbar -- the statistic the per-message decision would use
 * now: vbar = the mean of the server's v over all P parameters (a
 * compensated sum in a fixed order, rounded once to fp32), written to
 * vbar_dev (device float) on the handle's stream.  No draw is consumed and
 * no counter advances.  Errors: EINVAL, ENOMEM, ECUDA.
 */
FASGD_API int bfasgd_message_vbar(fasgd_t* h, float* vbar_dev);

/*
 * Per-tensor B-FASGD under a bandwidth budget (Sec. 5, future work: decide
 * per tensor, and spread a fixed bandwidth budget over the tensors by their
 * statistics).  The paper gives no formula; the reading implemented:
 *   vbar_t  = mean of the server's v over tensor t (exact sum, rounded once);
 *   a_t     = fl(vbar_t + eps_b);
 *   E(x)    = sum_t floor(s_t * fl(a_t / fl(a_t + x)) * 2^32)   (integers;
 *             a term is 0 where a_t is not positive and finite);
 *   c       = the smallest non-negative float x (or +inf) with
 *             E(x) <= min(budget, P) * 2^32: the Eq. 9 threshold at which the
 *             expected number of parameters transmitted meets the budget;
 *   u_t     = top 24 bits of word (t mod 4) of Philox4x32-10 at counter
 *             (2^31 + t div 4, client + 2^31 * stream, n, n >> 32), key = seed
 *             (n: the client's push count for stream 0, fetch count for
 *             stream 1, which then advances);
 *   tensor t is transmitted iff u_t * fl(a_t + c) < a_t * 2^24 (Eq. 9,
 *             exact).  A tensor that is not transmitted is left as it is.
 * The expected count of transmitted parameters is E(c) 2^-32 (<= budget) up
 * to P 2^-24 (the 24-bit draw).  vbar_t is summed in a fixed order with
 * float-float pairs: it equals the correctly rounded mean unless that mean
 * lies within about 1e-12 (relative) of a rounding boundary of fp32.
 */
#define BFASGD_TMAX 4096                      /* tensors in one partition */

/*
 * bfasgd_set_tensors -- partition the parameters into T contiguous tensors:
 * tensor t covers [o_t, o_t + sizes[t]), o_0 = 0, o_{t+1} = o_t + sizes[t].
 * sizes: host int64[T], each >= 1, summing to P; 1 <= T <= BFASGD_TMAX.
 * Requires an empty queue; waits for the handle's stream; allocates small
 * device tables (a few bytes per tensor and per 8,192 parameters).
 * Errors: EINVAL, EAGAIN, ENOMEM, ECUDA.
 */
FASGD_API int bfasgd_set_tensors(fasgd_t* h, int32_t T, const int64_t* sizes);

/*
 * bfasgd_push_budget -- queue a per-tensor B-FASGD push: when it is applied
 * (in arrival order, by fasgd_apply_pending, as its own pass) the server
 * forms vbar_t from its v at that moment, solves for c from `budget`
 * (expected parameters per push, >= 0; budget >= P sends every tensor),
 * decides each tensor, and applies Eq. 4-8 (or Eq. 1-2) with the push's
 * alpha(tau) to every parameter of the transmitted tensors, reading grad
 * there only.  grad: device fp32[P], 16-byte aligned, borrowed until the
 * apply completes.  Outputs written on the stream at the apply, each may be
 * NULL: sent_dev (device uint8[T], 1 = transmitted), c_dev (device float),
 * count_dev (device int64, parameters transmitted).
 * Errors: EINVAL (no partition, bad pointer, budget < 0), ERANGE, EAGAIN.
 */
FASGD_API int bfasgd_push_budget(fasgd_t* h, int32_t client, int64_t timestamp,
                                 const float* grad, int64_t budget, uint8_t* sent_dev,
                                 float* c_dev, int64_t* count_dev);

/*
 * bfasgd_fetch_budget -- per-tensor B-FASGD fetch, taken on the stream
 * against the current server state: the same rule with stream 1 and the
 * client's fetch count; the transmitted tensors of theta are copied into
 * theta_client (device fp32[P], 16-byte aligned), the rest of the client's
 * copy is left as it is.  Outputs as for bfasgd_push_budget.
 * Errors: EINVAL, ERANGE, ECUDA.
 */
FASGD_API int bfasgd_fetch_budget(fasgd_t* h, int32_t client, float* theta_client,
                                  int64_t budget, uint8_t* sent_dev, float* c_dev,
                                  int64_t* count_dev);

/*
 * fasgd_pull -- copy theta (P fp32) into params (host or device) and return
 * the server timestamp T in *T (Sec. 2.1 protocol step 3: the parameters
 * handed back to a client).  The copy is ordered after earlier work on the
 * handle's stream and later work on that stream waits for it (it runs on an
 * internal stream beside pending host-push copies).  Pending pushes are not
 * applied.
 * Either output may be NULL.  Errors: EINVAL, ECUDA.
 */
FASGD_API int fasgd_pull(fasgd_t* h, float* params, int64_t* T);

/*
 * fasgd_get_state / fasgd_set_state -- checkpoint and restore theta, n, b, v
 * (P fp32 each; host or device; any may be NULL to skip it) and T.
 * Both require an empty queue.  get_state blocks until the copies are done.
 * Errors: EINVAL, EAGAIN (pushes pending), ECUDA.
 */
FASGD_API int fasgd_get_state(fasgd_t* h, float* theta, float* n, float* b, float* v, int64_t* T);
FASGD_API int fasgd_set_state(fasgd_t* h, const float* theta, const float* n, const float* b,
                    const float* v, int64_t T);

/* Per-client B-FASGD push and fetch counters (lambda uint64 values, host memory). */
FASGD_API int fasgd_get_push_counts(fasgd_t* h, uint64_t* counts);
FASGD_API int fasgd_set_push_counts(fasgd_t* h, const uint64_t* counts);
FASGD_API int fasgd_get_fetch_counts(fasgd_t* h, uint64_t* counts);
FASGD_API int fasgd_set_fetch_counts(fasgd_t* h, const uint64_t* counts);

/*
 * fasgd_sync -- wait until the handle's stream is idle, then report and
 * clear the device-side error flags: FASGD_EDEVICE if a sparse list held a
 * bad entry, or a wait inside the dense pass's copy pipeline expired (it
 * gives up after about a second rather than hang), since the last sync;
 * else FASGD_OK (or ECUDA).
 */
FASGD_API int fasgd_sync(fasgd_t* h);

/*
 * fasgd_selftest_wait_expiry -- exercise the failure path of the dense pass's
 * copy pipeline (no counterpart in the paper): enqueue on the handle's
 * stream one small kernel whose pipeline barrier never completes.  Its two
 * bounded waits -- one thread and one whole warp, the forms the pass uses --
 * each give up after about a second and raise device flag 8, so the next
 * fasgd_sync returns FASGD_EDEVICE.  Changes no state; the handle stays
 * usable.  Errors: EINVAL, ECUDA.
 */
FASGD_API int fasgd_selftest_wait_expiry(fasgd_t* h);

/*
 * fasgd_selftest_fail_pass -- exercise the partial-failure path of
 * fasgd_apply_pending without any GPU fault: the pass of fasgd_apply_pending
 * that comes `after` passes from now (0: the next one) reports a launch
 * failure (ECUDA) instead of being launched; nothing runs on the GPU for it.
 * A pass is a fused run of dense pushes, a sparse push (one whose list is
 * known to be empty launches nothing and is not counted), or the update of a
 * message or budget push (after its decision).  after = -1 switches it off.
 * The paper has no counterpart; this is a test hook.  Errors: EINVAL.
 */
FASGD_API int fasgd_selftest_fail_pass(fasgd_t* h, int32_t after);

/* Server timestamp T (pushes applied so far) and number of queued pushes. */
FASGD_API int64_t fasgd_timestamp(const fasgd_t* h);
FASGD_API int64_t fasgd_pending(const fasgd_t* h);

/* Number of kernels this handle has launched since it was created. */
FASGD_API int64_t fasgd_kernel_launches(const fasgd_t* h);

/*
 * bfasgd_select_compact_noalloc -- the same send decision and compaction as
 * bfasgd_select_compact, for callers that cannot allocate device memory.
 * The paper has no counterpart; this entry point exists for deployment.
 *
 * Who needs it: code that may not call cudaMalloc when it runs -- for
 * example a host framework that owns every device allocation through its
 * own memory pool and forbids others, a process held to a fixed device
 * memory budget, or a latency-critical loop that cannot afford the implicit
 * device synchronisation an allocation can cause.  Such a caller cannot use
 * bfasgd_select_compact, because a handle allocates its state and scratch.
 *
 * This entry point needs no handle and allocates nothing.  Its scratch (the
 * per-parameter bit mask and the per-tile counts and offsets) lives in a
 * fixed static device array of BFASGD_NOALLOC_SCRATCH_BYTES (about 2 MiB)
 * that every GPU which loads the library holds until the process exits.
 * The first call on a device looks up that array's device address (once per
 * device, with that device current); make that first call before any
 * stream capture (a first call made while `stream` is capturing returns
 * FASGD_EINVAL and does nothing).  The address is kept for the life of the
 * process: after cudaDeviceReset on a device, do not call this entry point
 * on that device again.  All calls share the one array and the kernels
 * rewrite every scratch word before reading it, so nothing carries over
 * between calls -- but calls that overlap on the GPU (other streams, other
 * host threads) race on it and must be serialised by the caller.
 *
 * Arguments: P parameters, 1 <= P <= BFASGD_NOALLOC_PMAX (larger P is
 * rejected with FASGD_EINVAL and a message); grad and v: device fp32[P],
 * 16-byte aligned (v is the client's copy of the statistic; there is no
 * server here); c >= 0 (+inf allowed), eps_b finite >= 0; seed, client >= 0
 * and push_no form the Philox counter and key exactly as in
 * bfasgd_select_compact (push_no is the caller's per-client counter, not
 * advanced here); idx, val: device, room for P entries; n_dev: device int64;
 * stream: a cudaStream_t (NULL = legacy default stream).  Outputs as for
 * bfasgd_select_compact, written on the stream.
 * Errors: EINVAL (bad argument or P too large), ECUDA.
 */
#define BFASGD_NOALLOC_PMAX ((int64_t)1 << 24)              /* 16,777,216 parameters */
#define BFASGD_NOALLOC_SCRATCH_BYTES ((int64_t)2121728)     /* mask + tile counts + tile bases */
FASGD_API int bfasgd_select_compact_noalloc(int64_t P, const float* grad, const float* v, float c,
                                            float eps_b, uint64_t seed, int32_t client,
                                            uint64_t push_no, int32_t* idx, float* val,
                                            int64_t* n_dev, void* stream);

/*
 * Closed-loop simulation support (the paper's FRED simulator, Sec. 3, with a
 * synthetic objective in place of its MNIST model; no handle needed).
 *
 * fasgd_sim_quadratic_grad -- a client's stochastic gradient of
 * f(theta) = 1/2 sum_p h_p (theta_p - star_p)^2 at its copy theta:
 * grad_p = fl(fl(h_p (theta_p - star_p)) + fl(sigma_p xi_p)), xi_p uniform
 * with unit variance, xi_p = fl(((u + 1/2) 2^-23 - 1/2) * fl(sqrt 12)), u the
 * top 23 bits of word (p mod 4) of Philox4x32-10 at counter
 * (p div 4, client + 2^30, n, n >> 32), key = seed (n: the client's gradient
 * count).  All pointers device fp32[P], 16-byte aligned; 0 <= client < 2^30.
 * fasgd_sim_quadratic_loss -- *loss (device double) = f(theta), terms in
 * fp32 summed in a fixed order (reproducible); scratch: device, >= 1024
 * doubles.  Both run on `stream` (cudaStream_t, NULL = legacy default).
 * Errors: EINVAL (text via fasgd_last_error(NULL)), ECUDA.
 */
FASGD_API int fasgd_sim_quadratic_grad(int64_t P, const float* theta, const float* h,
                                       const float* star, const float* sigma, uint64_t seed,
                                       int32_t client, uint64_t n, float* grad, void* stream);
FASGD_API int fasgd_sim_quadratic_loss(int64_t P, const float* theta, const float* h,
                                       const float* star, double* scratch, double* loss,
                                       void* stream);

/* Text of the last failure on h, or, when h is NULL, of the last failed call
 * made without a handle (fasgd_create, bfasgd_fetch_apply, fasgd_sim_*,
 * bfasgd_select_compact_noalloc). */
FASGD_API const char* fasgd_last_error(const fasgd_t* h);

#ifdef __cplusplus
}
#endif

#endif /* FASGD_H */
