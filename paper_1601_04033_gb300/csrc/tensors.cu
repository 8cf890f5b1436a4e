// Per-tensor B-FASGD under a bandwidth budget (the paper's future-work
// section: decide per tensor, and spread a fixed bandwidth budget over the
// tensors according to their statistics).
//
// One decision takes one or two kernels:
//   1. tensor_partial (only when the item sums are stale): one block per
//      work item (a piece of one tensor of at most tensor_chunk(P)
//      parameters) sums v over the item -- per thread an fp32 sum with its
//      exact rounding errors (TwoSum), then a fixed float-float tree -- into
//      one float-float pair per item;
//   2. budget_resolve (one block of 1024 threads): vbar_t = fl32(sum of the
//      item sums of tensor t / s_t) for the tensors whose v changed since the
//      last decision (the others keep their cached vbar_t), the budget
//      threshold c, then the Philox draw and the exact Eq. 9 decision of
//      every tensor and the number of parameters transmitted.
// Then tensor_apply (a push: Eq. 4-8, or Eq. 1-2, on the transmitted
// tensors) or tensor_copy (a fetch: theta into the client's copy) walks the
// items of the transmitted tensors; the others cost one flag read.  The
// apply re-forms the sums of the items it rewrote, in the partial kernel's
// element order, so the item sums stay those of the current v and the next
// decision skips the partial kernel (the host tracks when another pass has
// changed v and the sums must be formed afresh).  All four are launched as
// programmatic dependents (pdl.cuh), so each one's launch overlaps the tail
// of the kernel before it.
//
// The threshold.  With a_t = fl(vbar_t + eps_b) and
//   E(x) = sum_t floor(s_t * fl(a_t / fl(a_t + x)) * 2^32),
// c is the smallest non-negative float x (or +inf) with E(x) <= limit.
// Every term is an integer and non-increasing in x (IEEE rounding is
// monotone), so E is exact in any summation order and the search has one
// answer.  The block searches the bit patterns of the non-negative floats
// (ordered as their values): each round evaluates E at 2^m - 1 points of
// the current interval, one group of warps per point (lanes over tensors,
// then an exact integer sum), and keeps the part between the last failing
// and the first passing point; the first round is centred on the previous
// threshold of the same stream, since the statistics move little per call.

#include "eq9.cuh"
#include "kernels.cuh"
#include "pdl.cuh"
#include "tensors.cuh"
#include "twosum.cuh"
#include "update.cuh"

namespace fasgd {
namespace {

constexpr int kItemThreads = 256;
constexpr unsigned kFull = 0xffffffffu;
constexpr int kTermsPerThread = 2;  // budget terms per thread and search round

// Exact sum over the warp of one 64-bit value per lane, from three 32-bit
// hardware reductions of 21-, 21- and 22-bit pieces (a sum of 32 pieces
// stays below 2^27, so none of them wraps).  The total must fit in 64 bits.
__device__ __forceinline__ unsigned long long warp_sum_u64(unsigned long long x) {
    const unsigned p0 = __reduce_add_sync(kFull, (unsigned)(x & 0x1fffffu));
    const unsigned p1 = __reduce_add_sync(kFull, (unsigned)((x >> 21) & 0x1fffffu));
    const unsigned p2 = __reduce_add_sync(kFull, (unsigned)(x >> 42));
    return (unsigned long long)p0 + ((unsigned long long)p1 << 21) + ((unsigned long long)p2 << 42);
}

// The sum of v over one item as a float-float pair, the same bits wherever
// it is formed (the partial kernel, or the apply kernel after it rewrote the
// item): thread tid adds, in this order and with TwoSum, the head element
// s + tid (before the first whole 16-byte quad), the tail element 4 qe + tid
// (after the last), then quads qs + tid, qs + tid + 256, ...; the threads'
// pairs go through a fixed float-float tree.  Four quads are loaded before
// they are added, so a thread keeps four loads in flight.  Called by every
// thread of the block; the result is valid in thread 0.  Plain loads (no
// read-only path): the apply kernel reads values it has just written.
__device__ float2 item_v_sum(const TensorItem& it, const float* v, float2* smem) {
    const int tid = threadIdx.x;
    const int64_t s = it.start, e = s + it.len;
    const int64_t qs = (s + 3) >> 2, qe = e >> 2;   // whole quads inside [s, e)
    float hi = 0.f, lo = 0.f;
    if (4 * qs >= e) {
        for (int64_t p = s + tid; p < e; p += kItemThreads) two_sum_acc(hi, lo, v[p]);
    } else {
        if (tid < 4 * qs - s) two_sum_acc(hi, lo, v[s + tid]);
        if (tid < e - 4 * qe) two_sum_acc(hi, lo, v[4 * qe + tid]);
        const float4* v4 = reinterpret_cast<const float4*>(v);
        for (int64_t q = qs + tid; q < qe; q += 4 * kItemThreads) {
            float4 x[4];
#pragma unroll
            for (int k = 0; k < 4; ++k)
                if (q + k * kItemThreads < qe) x[k] = v4[q + k * kItemThreads];
#pragma unroll
            for (int k = 0; k < 4; ++k)
                if (q + k * kItemThreads < qe) {
                    two_sum_acc(hi, lo, x[k].x);
                    two_sum_acc(hi, lo, x[k].y);
                    two_sum_acc(hi, lo, x[k].z);
                    two_sum_acc(hi, lo, x[k].w);
                }
        }
    }
    float h, l;
    two_sum(hi, lo, h, l);
    ff_warp_sum(h, l);
    if ((tid & 31) == 0) smem[tid >> 5] = make_float2(h, l);
    __syncthreads();
    float2 sum = make_float2(0.f, 0.f);
    if (tid == 0)
        for (int w = 0; w < kItemThreads / 32; ++w) ff_add(sum.x, sum.y, smem[w].x, smem[w].y);
    __syncthreads();
    return sum;
}

__global__ void __launch_bounds__(kItemThreads) tensor_partial_kernel(const __grid_constant__ TensorArgs a) {
    __shared__ float2 smem[kItemThreads / 32];
    pdl_wait();
    pdl_trigger();
    for (int64_t i = blockIdx.x; i < a.n_items; i += gridDim.x) {
        const float2 sum = item_v_sum(a.items[i], a.v, smem);
        if (threadIdx.x == 0) a.partial[i] = sum;
    }
}

// floor(size * q * 2^32) for q = fl(a / fl(a + x)), a = fl(vbar + eps_b),
// exactly: q = M 2^e with M its 24-bit significand, so the term is
// size * M shifted by e + 32 (q <= 1 keeps it at most size * 2^32).  The
// caller passes a = 0 where fl(vbar + eps_b) is not a positive finite
// number: such a tensor's term is 0.
__device__ __forceinline__ uint64_t budget_term(int32_t size, float a, float x) {
    if (!(a > 0.f)) return 0;
    const float q = __fdiv_rn(a, __fadd_rn(a, x));
    const uint32_t bits = __float_as_uint(q);     // q in [0, 1]: sign bit clear
    if (bits == 0) return 0;
    const uint32_t ex = bits >> 23;
    const uint64_t M = ex ? ((bits & 0x7fffffu) | 0x800000u) : (bits & 0x7fffffu);
    const int shift = (ex ? (int)ex : 1) - 150 + 32;
    const uint64_t prod = (uint64_t)(uint32_t)size * M;
    if (shift >= 0) return prod << shift;
    return shift > -64 ? prod >> (-shift) : 0;
}

// Candidate k (0 .. 2^m - 2) of a search round inside the open interval
// (lo, hi) of bit patterns: 2^m - 1 points cutting it into 2^m near-equal
// parts (consecutive patterns once the interval is short); values >= hi are
// not evaluated.
__device__ __forceinline__ long long candidate(long long lo, long long hi, int k, int m) {
    const long long span = hi - lo;
    return span <= (1ll << m) ? lo + 1 + k : lo + ((span * (k + 1)) >> m);
}

// Candidate k of a first round centred on the previous threshold's bit
// pattern cp (the statistics move little between calls): cp itself and
// cp -/+ 2^s for s growing to 18 (about 3 % of the value), non-decreasing in
// k; if c has moved further, the round still leaves a valid, wider interval.
__device__ __forceinline__ long long warm_candidate(long long cp, int k, int m) {
    const int h = (1 << (m - 1)) - 1;
    const int j = k - h;
    if (j == 0) return cp;
    const int aj = j < 0 ? -j : j;
    const long long off = 1ll << ((18 * aj + (h >> 1)) / h);
    const long long c = j < 0 ? cp - off : cp + off;
    return c < 0 ? 0 : (c > 0x7f800000 ? 0x7f800000 : c);
}

__global__ void __launch_bounds__(kTensorResolveThreads) budget_resolve_kernel(const __grid_constant__ TensorArgs a) {
    // Dynamic shared memory (tensor_resolve_smem): the item sums, the tensor
    // sums, vbar_t, a_t, the item ranges, the sizes and the stale flags; the
    // inputs are loaded once, four per thread in flight together.
    extern __shared__ __align__(16) unsigned char dsm[];
    float2* s_part = reinterpret_cast<float2*>(dsm);
    float2* s_sum = s_part + a.n_items;
    float* s_vbar = reinterpret_cast<float*>(s_sum + a.T);
    float* s_a = s_vbar + a.T;    // fl(vbar_t + eps_b), 0 where not positive and finite
    int32_t* s_begin = reinterpret_cast<int32_t*>(s_a + a.T);
    int32_t* s_size = s_begin + a.T + 1;
    uint8_t* s_dirty = reinterpret_cast<uint8_t*>(s_size + a.T);
    __shared__ unsigned long long s_e[32];
    __shared__ long long s_cand[32];   // this round's candidates (lanes >= ncand: hi)
    __shared__ long long s_lo, s_hi, s_cp;
    __shared__ unsigned long long s_count;
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    pdl_wait();
    pdl_trigger();
    // Loads in passes of four per thread, every load of a pass issued before
    // any of its stores to shared memory.
    const long long cp_in = tid == 0 ? *a.c_prev : 0;
    const int nload = a.n_items > a.T + 1 ? a.n_items : a.T + 1;
    constexpr int kPass = 4;
    for (int i0 = 0; i0 < nload; i0 += kPass * kTensorResolveThreads) {
        float2 pv[kPass];
        int32_t bg[kPass], sz[kPass];
        uint8_t dt[kPass];
        float vb[kPass];
#pragma unroll
        for (int u = 0; u < kPass; ++u) {
            const int i = i0 + u * kTensorResolveThreads + tid;
            pv[u] = make_float2(0.f, 0.f);
            bg[u] = 0;
            sz[u] = 0;
            dt[u] = 1;
            vb[u] = 0.f;
            if (i < a.n_items) pv[u] = a.partial[i];
            if (i <= a.T) bg[u] = a.item_begin[i];
            if (i < a.T) {
                sz[u] = a.sizes[i];
                vb[u] = a.vbar_cache[i];
                if (!a.all_dirty) dt[u] = a.dirty[i];
            }
        }
#pragma unroll
        for (int u = 0; u < kPass; ++u) {
            const int i = i0 + u * kTensorResolveThreads + tid;
            if (i < a.n_items) s_part[i] = pv[u];
            if (i <= a.T) s_begin[i] = bg[u];
            if (i < a.T) {
                s_size[i] = sz[u];
                s_vbar[i] = vb[u];
                s_dirty[i] = dt[u];
            }
        }
    }
    if (tid == 0) {
        s_count = 0;
        s_cp = cp_in;
    }
    __syncthreads();
    // vbar_t of every tensor whose v changed since it was last formed: warp
    // (t mod 32) adds its item sums (lanes over the items, then a fixed
    // shuffle tree, all in float-float); then thread t divides (ff_div_int).
    // The other tensors keep the cached value -- the same bits, since the
    // item sums are.
    for (int t = warp; t < a.T; t += 32) {
        if (!s_dirty[t]) continue;
        float h = 0.f, l = 0.f;
        for (int i = s_begin[t] + lane; i < s_begin[t + 1]; i += 32)
            ff_add(h, l, s_part[i].x, s_part[i].y);
        ff_warp_sum(h, l);
        if (lane == 0) s_sum[t] = make_float2(h, l);
    }
    __syncthreads();
    for (int t = tid; t < a.T; t += kTensorResolveThreads) {
        float vb = s_vbar[t];
        if (s_dirty[t]) {
            const float2 p = s_sum[t];
            vb = ff_div_int(p.x, p.y, s_size[t]);
            s_vbar[t] = vb;
            a.vbar_cache[t] = vb;
            a.dirty[t] = 0;
        }
        const float at = __fadd_rn(vb, a.eps_b);
        s_a[t] = at > 0.f && at != __int_as_float(0x7f800000) ? at : 0.f;
    }
    __syncthreads();
    // Invariant: E(lo) > limit >= E(hi) (lo = -1 stands below 0, hi = +inf
    // has E = 0); c = hi once they are adjacent.  2^m is chosen so that a
    // thread takes at most kTermsPerThread tensors per round: more candidates
    // per round mean fewer rounds, but every round's terms are issued by the
    // one SM.  Warp 0 places the candidates and takes each round's decision;
    // the other warps only evaluate terms.
    int m = 5;
    while (m > 1 && (a.T << m) > kTermsPerThread * kTensorResolveThreads) --m;
    const int gwarps = 32 >> m;                      // warps per group; the last group idles
    const int group = warp / gwarps;
    const int gthread = tid - group * gwarps * 32;
    const int gsize = gwarps * 32;
    const int ncand = (1 << m) - 1;
    // Warp 0 also keeps E at both ends of the interval (E(+inf) = 0; E at
    // lo = -1 unknown).  Once both are known, the next round's candidates
    // sit on a ladder (0, +-1, +-4, +-16, ...) around the point where the
    // straight line between them crosses the limit: E is smooth and the
    // interval short, so the crossing is usually within an ulp or two.  A
    // round placed that way that shrinks the interval less than an even
    // split would is followed by an even split, so the search always ends.
    long long w_elo = -1, w_ehi = 0, w_prev_span = 0;   // E(lo) (-1: unknown), E(hi)
    bool w_interp = false;
    if (warp == 0) {
        const long long cp = s_cp;
        const bool warm = m >= 3 && cp >= 0 && cp <= 0x7f800000;
        long long cand = 0x7f800000;
        if (lane < ncand) cand = warm ? warm_candidate(cp, lane, m) : candidate(-1, 0x7f800000, lane, m);
        s_cand[lane] = cand < 0x7f800000 ? cand : 0x7f800000;
        if (lane == 0) {
            s_lo = -1;
            s_hi = 0x7f800000;
        }
    }
    __syncthreads();
    long long lo = -1, hi = 0x7f800000;
    // At most 31 even splits with one candidate each (2^31 patterns), each
    // possibly preceded by one placed round: the cap is never reached.
    for (int round = 0; round < 128 && hi - lo > 1; ++round) {
        unsigned long long e = 0;
        const long long cand = s_cand[group < 32 ? group : 31];
        if (group < ncand && cand < hi) {
            // Two tensors at a time with separate sums, so that the two
            // divisions overlap.
            const float x = __uint_as_float((uint32_t)cand);
            unsigned long long e1 = 0;
            int t = gthread;
            for (; t + gsize < a.T; t += 2 * gsize) {
                e += budget_term(s_size[t], s_a[t], x);
                e1 += budget_term(s_size[t + gsize], s_a[t + gsize], x);
            }
            if (t < a.T) e += budget_term(s_size[t], s_a[t], x);
            e += e1;
        }
        e = warp_sum_u64(e);
        if (lane == 0) s_e[warp] = e;
        __syncthreads();
        if (warp == 0) {
            // Lane k adds the partials of group k and tests candidate k; E is
            // non-increasing and the candidates non-decreasing, so the passing
            // candidates are a suffix.  Then the next round's candidates.
            const long long ck = s_cand[lane];
            const bool evaluated = lane < ncand && ck < hi;
            long long ek = 0;
            if (evaluated) {
                unsigned long long sum = 0;
                for (int w = 0; w < gwarps; ++w) sum += s_e[lane * gwarps + w];
                ek = (long long)sum;
            }
            const int ok = !evaluated || ek <= a.limit;
            const long long cv = evaluated ? ck : hi;
            const unsigned pass = __ballot_sync(kFull, ok);   // lanes >= ncand pass
            const int first = __ffs(pass) - 1;
            const long long c_first = __shfl_sync(kFull, cv, first);
            const long long e_first = __shfl_sync(kFull, ek, first);
            const bool first_eval = __shfl_sync(kFull, evaluated, first);
            const long long c_prev = __shfl_sync(kFull, cv, first > 0 ? first - 1 : 0);
            const long long e_prev = __shfl_sync(kFull, ek, first > 0 ? first - 1 : 0);
            const long long nlo = first > 0 ? c_prev : lo;
            const long long nhi = c_first;
            w_elo = first > 0 ? e_prev : w_elo;
            w_ehi = first_eval ? e_first : w_ehi;
            const long long span = nhi - nlo;
            const bool interp = w_elo >= 0 && span > (1ll << m) &&
                                (!w_interp || (span << m) <= w_prev_span);
            long long nc;
            if (interp) {
                // f in (0, 1] only guides where the candidates go, so fp32
                // does (fp64 is a slow pipe here, on the round's critical path).
                const float f = (float)(w_elo - a.limit) / (float)(w_elo - w_ehi);
                long long xs = nlo + (long long)(f * (float)span);
                xs = xs <= nlo ? nlo + 1 : (xs >= nhi ? nhi - 1 : xs);
                const int h = (1 << (m - 1)) - 1;
                const int j = lane - h;
                const int aj = j < 0 ? -j : j;
                const long long off = aj == 0 ? 0 : 1ll << (2 * (aj - 1) < 40 ? 2 * (aj - 1) : 40);
                nc = j < 0 ? xs - off : xs + off;
                nc = nc <= nlo ? nlo + 1 : nc;
            } else {
                nc = candidate(nlo, nhi, lane, m);
            }
            s_cand[lane] = lane < ncand && nc < nhi ? nc : nhi;
            w_interp = interp;
            w_prev_span = span;
            if (lane == 0) {
                s_lo = nlo;
                s_hi = nhi;
            }
        }
        __syncthreads();
        lo = s_lo;
        hi = s_hi;
    }
    const float c = __uint_as_float((uint32_t)hi);
    // Whole warps walk the tensors (the count is summed with a shuffle).
    for (int t0 = tid - lane; t0 < a.T; t0 += kTensorResolveThreads) {
        const int t = t0 + lane;
        unsigned long long n = 0;
        if (t < a.T) {
            const Philox4 r = philox4x32_10(0x80000000u + ((uint32_t)t >> 2), a.client_word, a.n_lo,
                                            a.n_hi, a.round_key0, a.round_key1);
            const uint32_t u = (t & 2) ? ((t & 1) ? r.x[3] : r.x[2]) : ((t & 1) ? r.x[1] : r.x[0]);
            const uint32_t send = send_bit(u >> 8, s_vbar[t], c, a.eps_b);
            a.sent[t] = (uint8_t)send;
            if (a.user_sent != nullptr) a.user_sent[t] = (uint8_t)send;
            if (send && a.mark_dirty) a.dirty[t] = 1;    // the apply that follows rewrites its v
            n = send ? (unsigned long long)s_size[t] : 0ull;
        }
#pragma unroll
        for (int off = 16; off > 0; off >>= 1) n += __shfl_xor_sync(kFull, n, off);
        if (lane == 0 && n != 0) atomicAdd(&s_count, n);
    }
    __syncthreads();
    if (tid == 0) {
        *a.c_out = c;
        *a.count_out = (int64_t)s_count;
        *a.c_prev = hi;
        if (a.user_c != nullptr) *a.user_c = c;
        if (a.user_count != nullptr) *a.user_count = (int64_t)s_count;
    }
}

template <int RULE, int ARITH>
__device__ __forceinline__ void update4(float4& th, float4& n, float4& b, float4& v, const float4& g,
                                        float coef, const StatParams& sp) {
    if (RULE == kRuleSgd) {
        sgd_update(th.x, g.x, coef);
        sgd_update(th.y, g.y, coef);
        sgd_update(th.z, g.z, coef);
        sgd_update(th.w, g.w, coef);
    } else {
        constexpr bool STD = RULE == kRuleFasgdStd;
        rule_update<ARITH, STD>(th.x, n.x, b.x, v.x, g.x, coef, sp);
        rule_update<ARITH, STD>(th.y, n.y, b.y, v.y, g.y, coef, sp);
        rule_update<ARITH, STD>(th.z, n.z, b.z, v.z, g.z, coef, sp);
        rule_update<ARITH, STD>(th.w, n.w, b.w, v.w, g.w, coef, sp);
    }
}

template <int RULE, int ARITH>
__device__ __forceinline__ void update1(const RangeArgs& a, int64_t p) {
    float th = a.theta[p];
    if (RULE == kRuleSgd) {
        sgd_update(th, a.grad[p], a.coef);
    } else {
        float n = a.n[p], b = a.b[p], v = a.v[p];
        rule_update<ARITH, RULE == kRuleFasgdStd>(th, n, b, v, a.grad[p], a.coef, a.sp);
        a.n[p] = n;
        a.b[p] = b;
        a.v[p] = v;
    }
    a.theta[p] = th;
}

__device__ __forceinline__ float4 ld4(const float* base, int64_t q) {
    return reinterpret_cast<const float4*>(base)[q];
}
__device__ __forceinline__ void st4(float* base, int64_t q, const float4& x) {
    reinterpret_cast<float4*>(base)[q] = x;
}

// Eq. 4-8 (or Eq. 1-2) on every parameter of the transmitted tensors.  The
// head and tail of an item (outside whole 16-byte quads) go element by
// element; the quads two per thread per step, loads before stores.  When
// partial is set (rules that change v), the block then re-forms the item's
// sum of v from the values it just wrote (from L2), with the same element
// order as the partial kernel, so the next decision needs no pass over v.
template <int RULE, int ARITH>
__global__ void __launch_bounds__(kItemThreads) tensor_apply_kernel(const __grid_constant__ RangeArgs a) {
    constexpr bool FAS = RULE != kRuleSgd;
    __shared__ float2 smem[kItemThreads / 32];
    const int tid = threadIdx.x;
    pdl_wait();
    pdl_trigger();
    for (int64_t i = blockIdx.x; i < a.n_items; i += gridDim.x) {
        const TensorItem it = a.items[i];
        if (!a.sent[it.tensor]) continue;
        const int64_t s = it.start, e = s + it.len;
        const int64_t qs = (s + 3) >> 2, qe = e >> 2;
        if (4 * qs >= e) {
            for (int64_t p = s + tid; p < e; p += kItemThreads) update1<RULE, ARITH>(a, p);
        } else {
            if (tid < 4 * qs - s) update1<RULE, ARITH>(a, s + tid);
            if (tid < e - 4 * qe) update1<RULE, ARITH>(a, 4 * qe + tid);
            for (int64_t q0 = qs + tid; q0 < qe; q0 += 2 * kItemThreads) {
                const int64_t q1 = q0 + kItemThreads;
                const bool two = q1 < qe;
                float4 th0, n0, b0, v0, g0, th1, n1, b1, v1, g1;
                g0 = __ldcs(reinterpret_cast<const float4*>(a.grad) + q0);
                th0 = ld4(a.theta, q0);
                if (FAS) {
                    n0 = ld4(a.n, q0);
                    b0 = ld4(a.b, q0);
                    v0 = ld4(a.v, q0);
                }
                if (two) {
                    g1 = __ldcs(reinterpret_cast<const float4*>(a.grad) + q1);
                    th1 = ld4(a.theta, q1);
                    if (FAS) {
                        n1 = ld4(a.n, q1);
                        b1 = ld4(a.b, q1);
                        v1 = ld4(a.v, q1);
                    }
                }
                update4<RULE, ARITH>(th0, n0, b0, v0, g0, a.coef, a.sp);
                st4(a.theta, q0, th0);
                if (FAS) {
                    st4(a.n, q0, n0);
                    st4(a.b, q0, b0);
                    st4(a.v, q0, v0);
                }
                if (two) {
                    update4<RULE, ARITH>(th1, n1, b1, v1, g1, a.coef, a.sp);
                    st4(a.theta, q1, th1);
                    if (FAS) {
                        st4(a.n, q1, n1);
                        st4(a.b, q1, b1);
                        st4(a.v, q1, v1);
                    }
                }
            }
        }
        if (FAS && a.partial != nullptr) {
            __syncthreads();    // the block's writes of v are visible to the block
            const float2 sum = item_v_sum(it, a.v, smem);
            if (tid == 0) a.partial[i] = sum;
        }
    }
}

// dst <- src on every parameter of the transmitted tensors, eight quads per
// thread in flight.
__global__ void __launch_bounds__(kItemThreads) tensor_copy_kernel(const __grid_constant__ RangeArgs a) {
    const int tid = threadIdx.x;
    pdl_wait();
    pdl_trigger();
    for (int64_t i = blockIdx.x; i < a.n_items; i += gridDim.x) {
        const TensorItem it = a.items[i];
        if (!a.sent[it.tensor]) continue;
        const int64_t s = it.start, e = s + it.len;
        const int64_t qs = (s + 3) >> 2, qe = e >> 2;
        if (4 * qs >= e) {
            for (int64_t p = s + tid; p < e; p += kItemThreads) a.dst[p] = a.src[p];
            continue;
        }
        if (tid < 4 * qs - s) a.dst[s + tid] = a.src[s + tid];
        if (tid < e - 4 * qe) a.dst[4 * qe + tid] = a.src[4 * qe + tid];
        for (int64_t q = qs + tid; q < qe; q += 8 * kItemThreads) {
            float4 x[8];
#pragma unroll
            for (int k = 0; k < 8; ++k)
                if (q + k * kItemThreads < qe) x[k] = ld4(a.src, q + k * kItemThreads);
#pragma unroll
            for (int k = 0; k < 8; ++k)
                if (q + k * kItemThreads < qe) st4(a.dst, q + k * kItemThreads, x[k]);
        }
    }
}

unsigned item_grid(int32_t n_items) { return (unsigned)(n_items > 0 ? n_items : 1); }

template <int RULE, int ARITH>
cudaError_t launch_apply_rule(const RangeArgs& a, cudaStream_t stream) {
    return launch_pdl(tensor_apply_kernel<RULE, ARITH>, item_grid(a.n_items), kItemThreads, 0,
                      stream, a);
}

}  // namespace

cudaError_t launch_tensor_decide(const TensorArgs& a, bool sums_valid, cudaStream_t stream,
                                 int64_t* launches) {
    cudaError_t st;
    if (!sums_valid) {
        st = launch_pdl(tensor_partial_kernel, item_grid(a.n_items), kItemThreads, 0, stream, a);
        if (st != cudaSuccess) return st;
        ++*launches;
    }
    const size_t smem = tensor_resolve_smem(a.n_items, a.T);
    st = cudaFuncSetAttribute(budget_resolve_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                              (int)smem);
    if (st != cudaSuccess) return st;
    st = launch_pdl(budget_resolve_kernel, 1, kTensorResolveThreads, smem, stream, a);
    if (st == cudaSuccess) ++*launches;
    return st;
}

cudaError_t launch_tensor_apply(const RangeArgs& a, int rule, bool exact, cudaStream_t stream,
                                int64_t* launches) {
    const bool ftz = a.sp.eps >= kFtzSafeEps;
    cudaError_t st;
    if (rule == kRuleSgd)
        st = launch_apply_rule<kRuleSgd, kArithApprox>(a, stream);
    else if (rule == kRuleFasgd)
        st = exact ? launch_apply_rule<kRuleFasgd, kArithExact>(a, stream)
             : ftz ? launch_apply_rule<kRuleFasgd, kArithApproxFtz>(a, stream)
                   : launch_apply_rule<kRuleFasgd, kArithApprox>(a, stream);
    else
        st = exact ? launch_apply_rule<kRuleFasgdStd, kArithExact>(a, stream)
             : ftz ? launch_apply_rule<kRuleFasgdStd, kArithApproxFtz>(a, stream)
                   : launch_apply_rule<kRuleFasgdStd, kArithApprox>(a, stream);
    if (st == cudaSuccess) ++*launches;
    return st;
}

cudaError_t launch_tensor_copy(const RangeArgs& a, cudaStream_t stream, int64_t* launches) {
    cudaError_t st = launch_pdl(tensor_copy_kernel, item_grid(a.n_items), kItemThreads, 0, stream, a);
    if (st == cudaSuccess) ++*launches;
    return st;
}

}  // namespace fasgd
