/*
 * FASGD / SASGD / ASGD / B-FASGD reference oracle -- TEST INFRASTRUCTURE ONLY.
 *
 * A plain, slow, single-threaded restatement of the update rules of
 * "Faster Asynchronous SGD" (Odena, 2016), written to check the CUDA path.
 * Only the tests, the smoke check and the CPU-baseline leg of the benchmark
 * load it; the product path never does.  It shares no code, header, table or
 * constant with the CUDA path.
 *
 * Precision: REAL is the type of the parameters and statistics.  The build
 * makes two copies: REAL=float (the fp32 parameters and state the server
 * keeps; every operation rounded once, IEEE round-to-nearest, compiled with
 * -ffp-contract=off so nothing is fused) and REAL=double (the same rules in
 * fp64, the exact-arithmetic yardstick for drift).  The B-FASGD send
 * decision is always taken in fp32, the precision the kernel takes it in.
 *
 * Every function is elementwise over the parameter vector and follows the
 * paper's order of operations:
 *   Eq. 1-2  (Sec. 2.1)  g = alpha(tau) * dtheta,  theta <- theta - g
 *   Eq. 4-6  (Sec. 2.2)  n, b moving averages; v moving average of 1/std
 *   Eq. 7-8  (Sec. 2.2)  theta <- theta - alpha / (v * tau) * dtheta
 *   Eq. 9    (Sec. 2.3)  transmit (push or fetch) iff r < 1 / (1 + c / (v + eps))
 * Readings where the paper is silent:
 *   tau = 0 divides by zero in Eq. 1 and Eq. 7: the divisor is max(tau, 1);
 *   n - b^2 can round below zero in floating point: it is clamped at 0
 *   before eps is added (a no-op in exact arithmetic);
 *   the step of Eq. 7 uses the v just updated by Eq. 6 (subscript i);
 *   Eq. 9 is applied per parameter with that parameter's own v_p, and r is
 *   u / 2^24 for a 24-bit counter-based draw u, compared strictly.
 */
#include <math.h>
#include <stdint.h>
#include <string.h>

#ifndef REAL
#define REAL float
#endif

#define ORA_ASGD 0
#define ORA_SASGD 1
#define ORA_FASGD 2
#define ORA_FASGD_STD 3

/* Size of REAL, so the Python side can check which build it loaded. */
int ora_real_bytes(void) { return (int)sizeof(REAL); }

/*
 * Per-push learning-rate factor alpha(tau) of Eq. 1 and alpha / tau of
 * Eq. 7 (the division by v is per element, in the step).  ASGD uses the
 * master rate alone (the protocol of Sec. 2.1).  The quotient is formed in
 * fp64 and rounded once to REAL.
 */
REAL ora_coef(int variant, float alpha, int64_t tau)
{
    if (variant == ORA_ASGD)
        return (REAL)alpha;
    int64_t t = tau < 1 ? 1 : tau;
    return (REAL)((double)alpha / (double)t);
}

static REAL ora_sqrt(REAL x)
{
    return sizeof(REAL) == sizeof(float) ? (REAL)sqrtf((float)x) : (REAL)sqrt((double)x);
}

static REAL ora_max0(REAL x)
{
    return sizeof(REAL) == sizeof(float) ? (REAL)fmaxf((float)x, 0.0f) : (REAL)fmax((double)x, 0.0);
}

/*
 * One server update of one parameter with gradient entry g.
 * FASGD: Eq. 4, Eq. 5, Eq. 6, then Eq. 7-8 with the new v.
 * ASGD / SASGD: Eq. 1-2 (the statistics are not touched).
 */
static void ora_update_one(int variant, REAL *theta, REAL *n, REAL *b, REAL *v,
                           REAL g, REAL coef, REAL gamma, REAL beta, REAL eps)
{
    if (variant == ORA_FASGD) {
        *n = gamma * *n + (1 - gamma) * (g * g);          /* Eq. 4 */
        *b = gamma * *b + (1 - gamma) * g;                /* Eq. 5 */
        REAL var = ora_max0(*n - *b * *b);
        REAL r = 1 / ora_sqrt(var + eps);
        *v = beta * *v + (1 - beta) * r;                  /* Eq. 6 */
        *theta = *theta - coef * g / *v;                  /* Eq. 7-8 */
    } else if (variant == ORA_FASGD_STD) {
        /* The prose reading of Sec. 2.2 ("dividing the learning rate by the
         * standard deviation"): v averages the std itself, and Eq. 7 divides
         * by it. */
        *n = gamma * *n + (1 - gamma) * (g * g);
        *b = gamma * *b + (1 - gamma) * g;
        REAL var = ora_max0(*n - *b * *b);
        REAL r = ora_sqrt(var + eps);
        *v = beta * *v + (1 - beta) * r;
        *theta = *theta - coef * g / *v;
    } else {
        *theta = *theta - coef * g;                       /* Eq. 1-2 */
    }
}

/* One dense push: every parameter p in [0, P) receives g[p]. */
void ora_apply_dense(int variant, int64_t P, REAL *theta, REAL *n, REAL *b, REAL *v,
                     const float *g, REAL coef, REAL gamma, REAL beta, REAL eps)
{
    for (int64_t p = 0; p < P; p++)
        ora_update_one(variant, &theta[p], &n[p], &b[p], &v[p], (REAL)g[p], coef,
                       gamma, beta, eps);
}

/*
 * One sparse push: parameter idx[i] receives val[i] for i < count; every
 * other parameter is left as it is (no decay of its statistics).
 * Returns 0, or -1 (and applies nothing) if an index is out of range or
 * the list is not strictly ascending.
 */
int ora_apply_sparse(int variant, int64_t P, REAL *theta, REAL *n, REAL *b, REAL *v,
                     int64_t count, const int32_t *idx, const float *val, REAL coef,
                     REAL gamma, REAL beta, REAL eps)
{
    for (int64_t i = 0; i < count; i++) {
        if (idx[i] < 0 || idx[i] >= P)
            return -1;
        if (i > 0 && idx[i] <= idx[i - 1])
            return -1;
    }
    for (int64_t i = 0; i < count; i++) {
        int64_t p = idx[i];
        ora_update_one(variant, &theta[p], &n[p], &b[p], &v[p], (REAL)val[i], coef,
                       gamma, beta, eps);
    }
    return 0;
}

/*
 * Philox4x32-10 (Salmon, Moraes, Dror, Shaw, "Parallel random numbers: as
 * easy as 1, 2, 3", SC'11): ten rounds of the Philox S-box on a 128-bit
 * counter under a 64-bit key, the key advanced by the Weyl increments
 * between rounds.
 */
static void ora_mulhilo(uint32_t a, uint32_t b, uint32_t *hi, uint32_t *lo)
{
    uint64_t prod = (uint64_t)a * (uint64_t)b;
    *hi = (uint32_t)(prod >> 32);
    *lo = (uint32_t)prod;
}

void ora_philox4x32_10(const uint32_t ctr_in[4], const uint32_t key_in[2], uint32_t out[4])
{
    const uint32_t mult0 = 0xD2511F53u, mult1 = 0xCD9E8D57u;
    const uint32_t weyl0 = 0x9E3779B9u, weyl1 = 0xBB67AE85u;
    uint32_t x0 = ctr_in[0], x1 = ctr_in[1], x2 = ctr_in[2], x3 = ctr_in[3];
    uint32_t k0 = key_in[0], k1 = key_in[1];
    for (int round = 0; round < 10; round++) {
        if (round > 0) {
            k0 += weyl0;
            k1 += weyl1;
        }
        uint32_t hi0, lo0, hi1, lo1;
        ora_mulhilo(mult0, x0, &hi0, &lo0);
        ora_mulhilo(mult1, x2, &hi1, &lo1);
        uint32_t y0 = hi1 ^ x1 ^ k0;
        uint32_t y1 = lo1;
        uint32_t y2 = hi0 ^ x3 ^ k1;
        uint32_t y3 = lo0;
        x0 = y0; x1 = y1; x2 = y2; x3 = y3;
    }
    out[0] = x0; out[1] = x1; out[2] = x2; out[3] = x3;
}

/*
 * The 24-bit uniform draw u_p for parameter p of one transmission.  The
 * counter is (p div 4, client + 2^31 * stream, n low word, n high word),
 * where n counts the client's earlier transmissions of that stream (stream
 * 0: pushes, stream 1: fetches); the key is the 64-bit seed; word (p mod 4)
 * of the Philox output is used, shifted down to its top 24 bits; r = u / 2^24
 * lies in [0, 1).
 */
uint32_t ora_draw_stream(uint64_t seed, uint32_t stream, uint32_t client, uint64_t push_no,
                         int64_t p)
{
    uint32_t ctr[4] = {(uint32_t)(p >> 2), client | (stream << 31), (uint32_t)push_no,
                       (uint32_t)(push_no >> 32)};
    uint32_t key[2] = {(uint32_t)seed, (uint32_t)(seed >> 32)};
    uint32_t out[4];
    ora_philox4x32_10(ctr, key, out);
    return out[p & 3] >> 8;
}

/* The push decisions use stream 0, the fetch decisions (below) stream 1. */
uint32_t ora_draw(uint64_t seed, uint32_t client, uint64_t push_no, int64_t p)
{
    return ora_draw_stream(seed, 0, client, push_no, p);
}

/*
 * Eq. 9 for one parameter, decided in fp32.  With a = fl(v + eps_b),
 * d = fl(a + c) and r = u / 2^24, and a, d > 0:
 *     r < 1 / (1 + c / a)  <=>  r < a / (a + c)  <=>  u * d < a * 2^24.
 * Both sides are formed in fp64, where they are exact: u has 24 bits and d
 * a 24-bit significand, so u * d has at most 48; a * 2^24 is a power-of-two
 * scaling, far inside fp64's exponent range.  (d = +inf never sends: the
 * product is +inf, or NaN for u = 0, and neither is below a finite bound.)
 * Returns 1 to transmit, 0 to drop.
 */
int ora_decide(uint32_t u, float v, float c, float eps_b)
{
    float a = v + eps_b;
    float d = a + c;
    return (double)u * (double)d < (double)a * 16777216.0;
}

/*
 * B-FASGD per-parameter push decision and compaction (Sec. 2.3, applied per
 * parameter as the paper's future-work section proposes): for p ascending,
 * keep p iff Eq. 9 holds for v[p]; write idx[m] = p and val[m] = g[p]
 * (bit copy).  Returns the number m of parameters kept.
 */
int64_t ora_select_stream(int64_t P, const float *g, const float *v, float c, float eps_b,
                          uint64_t seed, uint32_t stream, uint32_t client, uint64_t push_no,
                          int32_t *idx, float *val)
{
    int64_t m = 0;
    for (int64_t p = 0; p < P; p++) {
        uint32_t u = ora_draw_stream(seed, stream, client, push_no, p);
        if (ora_decide(u, v[p], c, eps_b)) {
            idx[m] = (int32_t)p;
            val[m] = g[p];
            m++;
        }
    }
    return m;
}

int64_t ora_select(int64_t P, const float *g, const float *v, float c, float eps_b,
                   uint64_t seed, uint32_t client, uint64_t push_no,
                   int32_t *idx, float *val)
{
    return ora_select_stream(P, g, v, c, eps_b, seed, 0, client, push_no, idx, val);
}

/*
 * B-FASGD fetch, per parameter (Sec. 2.3 applies Eq. 9 to each chance a
 * client has to receive fresh parameters; here per parameter, the extension
 * of the future-work section): the server keeps p iff Eq. 9 holds for v[p] with the
 * fetch threshold c (stream 1 draws) and sends (p, theta[p]); the client
 * overwrites its copy at the kept indices and keeps computing with its own
 * stale values everywhere else.
 */
int64_t ora_fetch_select(int64_t P, const float *theta, const float *v, float c, float eps_b,
                         uint64_t seed, uint32_t client, uint64_t fetch_no,
                         int32_t *idx, float *val)
{
    return ora_select_stream(P, theta, v, c, eps_b, seed, 1, client, fetch_no, idx, val);
}

void ora_fetch_apply(float *theta_client, int64_t count, const int32_t *idx, const float *val)
{
    for (int64_t i = 0; i < count; i++)
        theta_client[idx[i]] = val[i];
}

/*
 * Exact means, rounded once to fp32 (the statistic of the per-message and
 * per-tensor rules below).
 *
 * Every finite double is an integer multiple of 2^-1074 (its smallest
 * subnormal), and so is every float, so a sum of them is an integer number
 * of those units and can be formed with no rounding at all in a long
 * fixed-point accumulator (a Kulisch accumulator): ORA_LIMBS little-endian
 * 32-bit words, enough for 2^31 terms below 2^1024, one for the positive
 * and one for the negative terms.  The mean is the exact quotient of that
 * integer by the count, rounded to the nearest fp32 (ties to even).
 */
#define ORA_LIMBS 68

typedef struct {
    uint32_t pos[ORA_LIMBS], neg[ORA_LIMBS];
    int nan, pinf, ninf;
} ora_exact_sum;

static void ora_sum_clear(ora_exact_sum *s)
{
    memset(s, 0, sizeof *s);
}

/* w += m * 2^shift (m < 2^53, shift < 2046) */
static void ora_acc_add(uint32_t *w, uint64_t m, int shift)
{
    int i = shift / 32, bit = shift % 32;
    uint64_t lo = (m & 0xFFFFFFFFu) << bit;         /* < 2^63 */
    uint64_t hi = (m >> 32) << bit;                 /* < 2^52 */
    uint64_t c = (uint64_t)w[i] + (lo & 0xFFFFFFFFu);
    w[i] = (uint32_t)c;
    c = (c >> 32) + (uint64_t)w[i + 1] + (lo >> 32) + (hi & 0xFFFFFFFFu);
    w[i + 1] = (uint32_t)c;
    c = (c >> 32) + (uint64_t)w[i + 2] + (hi >> 32);
    w[i + 2] = (uint32_t)c;
    c >>= 32;
    for (int k = i + 3; c != 0 && k < ORA_LIMBS; k++) {
        c += w[k];
        w[k] = (uint32_t)c;
        c >>= 32;
    }
}

/* Adds x exactly: a finite double is m 2^(E-1075) for a normal encoding
 * (E = biased exponent, m = 2^52 + fraction) and fraction 2^-1074 for a
 * subnormal one, i.e. m units of 2^-1074 shifted left by max(E - 1, 0). */
static void ora_sum_add(ora_exact_sum *s, double x)
{
    uint64_t bits;
    memcpy(&bits, &x, sizeof bits);
    int neg = (int)(bits >> 63);
    int E = (int)((bits >> 52) & 0x7FF);
    uint64_t F = bits & (((uint64_t)1 << 52) - 1);
    if (E == 0x7FF) {                                /* inf or NaN: IEEE rules */
        if (F != 0)
            s->nan = 1;
        else if (neg)
            s->ninf = 1;
        else
            s->pinf = 1;
        return;
    }
    uint64_t m = E == 0 ? F : F | ((uint64_t)1 << 52);
    ora_acc_add(neg ? s->neg : s->pos, m, E == 0 ? 0 : E - 1);
}

static int ora_acc_cmp(const uint32_t *a, const uint32_t *b)
{
    for (int k = ORA_LIMBS - 1; k >= 0; k--)
        if (a[k] != b[k])
            return a[k] < b[k] ? -1 : 1;
    return 0;
}

/* The sum divided by count (1 <= count < 2^32), rounded to the nearest
 * float, ties to even. */
static float ora_sum_mean(const ora_exact_sum *s, int64_t count)
{
    if (s->nan || (s->pinf && s->ninf) || count < 1)
        return NAN;
    if (s->pinf)
        return INFINITY;
    if (s->ninf)
        return -INFINITY;
    /* |sum| = big - small, with the sign of the larger accumulator */
    int c = ora_acc_cmp(s->pos, s->neg);
    const uint32_t *big = c >= 0 ? s->pos : s->neg, *small = c >= 0 ? s->neg : s->pos;
    uint32_t q[ORA_LIMBS];
    int64_t borrow = 0;
    for (int k = 0; k < ORA_LIMBS; k++) {
        int64_t d = (int64_t)big[k] - (int64_t)small[k] - borrow;
        borrow = d < 0;
        q[k] = (uint32_t)(d + (borrow ? ((int64_t)1 << 32) : 0));
    }
    /* q <- floor(|sum| / count), r = the remainder (schoolbook, top down) */
    uint64_t r = 0;
    for (int k = ORA_LIMBS - 1; k >= 0; k--) {
        uint64_t cur = (r << 32) | q[k];
        q[k] = (uint32_t)(cur / (uint64_t)count);
        r = cur % (uint64_t)count;
    }
    /* Bit length L of q; the mean is (q + r / count) 2^-1074.  Its fp32
     * spacing is 2^(L - 1098) in the normal range and 2^-149 below it: in
     * units of 2^-1074, 2^shift with shift = max(L - 24, 925). */
    int L = 0;
    for (int k = ORA_LIMBS - 1; k >= 0 && L == 0; k--)
        for (int bit = 31; bit >= 0; bit--)
            if ((q[k] >> bit) & 1u) {
                L = 32 * k + bit + 1;
                break;
            }
    int shift = L - 24 > 925 ? L - 24 : 925;
    uint64_t mant = 0;                          /* q >> shift: at most 24 bits */
    for (int bit = shift + 23; bit >= shift; bit--)
        mant = (mant << 1) | ((q[bit / 32] >> (bit % 32)) & 1u);
    int guard = (q[(shift - 1) / 32] >> ((shift - 1) % 32)) & 1u;
    int sticky = r != 0;
    for (int bit = 0; bit < shift - 1 && !sticky; bit++)
        sticky = (q[bit / 32] >> (bit % 32)) & 1u;
    if (guard && (sticky || (mant & 1u)))
        mant++;
    float mag = ldexpf((float)mant, shift - 1074);   /* exact, or inf past FLT_MAX */
    return c >= 0 ? mag : -mag;
}

/*
 * The paper's literal B-FASGD (Sec. 2.3): one decision per transmission
 * opportunity, with v the mean over all parameters of the server's moving
 * averages.  ora_mean_v returns that mean: the exact sum of v divided by P,
 * rounded once to fp32.  The decision is Eq. 9 in fp32 (ora_decide) with a
 * draw from the message domain: word 0 of Philox4x32-10 at counter
 * (2^32 - 1, client + 2^31 * stream, n low, n high), top 24 bits (the
 * per-parameter draws never reach that first counter word, since
 * p div 4 < 2^29).
 */
float ora_mean_v(int64_t P, const REAL *v)
{
    ora_exact_sum s;
    ora_sum_clear(&s);
    for (int64_t p = 0; p < P; p++)
        ora_sum_add(&s, (double)v[p]);
    return ora_sum_mean(&s, P);
}

uint32_t ora_draw_message(uint64_t seed, uint32_t stream, uint32_t client, uint64_t n)
{
    uint32_t ctr[4] = {0xFFFFFFFFu, client | (stream << 31), (uint32_t)n, (uint32_t)(n >> 32)};
    uint32_t key[2] = {(uint32_t)seed, (uint32_t)(seed >> 32)};
    uint32_t out[4];
    ora_philox4x32_10(ctr, key, out);
    return out[0] >> 8;
}

/*
 * Closed-loop simulation (in the spirit of the paper's FRED simulator,
 * Sec. 3): clients compute stochastic gradients of a synthetic separable
 * quadratic f(theta) = 1/2 sum_p h_p (theta_p - star_p)^2 on their own
 * (stale) copies.  The gradient noise is uniform with variance sigma_p^2,
 * built from a 23-bit draw so that every operation is exact or rounded once
 * in fp32:
 *   u  = Philox word (p mod 4) at counter (p div 4, client + 2^30, n, n >> 32),
 *        top 23 bits (n = the client's gradient count);
 *   x  = (u + 1/2) 2^-23 - 1/2            (exact, in (-1/2, 1/2))
 *   xi = fl(x * fl(sqrt(12)))             (unit variance)
 *   g  = fl( fl(h (theta - star)) + fl(sigma xi) ).
 */
void ora_sim_grad(int64_t P, const float *theta, const float *h, const float *star,
                  const float *sigma, uint64_t seed, uint32_t client, uint64_t n, float *g)
{
    const float root12 = 3.46410161513775458705f;
    uint32_t key[2] = {(uint32_t)seed, (uint32_t)(seed >> 32)};
    for (int64_t p = 0; p < P; p++) {
        uint32_t ctr[4] = {(uint32_t)(p >> 2), client | (1u << 30), (uint32_t)n,
                           (uint32_t)(n >> 32)};
        uint32_t out[4];
        ora_philox4x32_10(ctr, key, out);
        uint32_t u = out[p & 3] >> 9;
        float x = ((float)u + 0.5f) * (1.0f / 8388608.0f) - 0.5f;
        float xi = x * root12;
        float d = theta[p] - star[p];
        g[p] = h[p] * d + sigma[p] * xi;
    }
}

/* f(theta) = 1/2 sum_p h_p (theta_p - star_p)^2, each term in fp32, summed in fp64. */
double ora_sim_loss(int64_t P, const float *theta, const float *h, const float *star)
{
    double s = 0.0;
    for (int64_t p = 0; p < P; p++) {
        float d = theta[p] - star[p];
        float t = h[p] * (d * d);
        s += (double)t;
    }
    return 0.5 * s;
}

/*
 * Per-tensor B-FASGD under a bandwidth budget (Sec. 5, future work: decide
 * per tensor rather than per message, and spread a fixed bandwidth budget
 * over the tensors according to their statistics).  The paper gives no
 * formula; the reading built here:
 *
 *   tensors    contiguous ranges [o_t, o_t + s_t) that partition [0, P),
 *              o_0 = 0, o_{t+1} = o_t + s_t, s_t >= 1;
 *   statistic  vbar_t = the mean of v over tensor t (exact sum, rounded
 *              once to fp32), as the per-message rule uses
 *              the mean over all parameters;
 *   decision   Eq. 9 per tensor: transmit tensor t iff
 *              u_t / 2^24 < 1 / (1 + c / (vbar_t + eps_b))   (ora_decide);
 *   budget     c is chosen so that the expected number of parameters
 *              transmitted does not exceed the budget B:
 *                  E(x) = sum_t floor(s_t * q_t(x) * 2^32),
 *                  q_t(x) = fl(a_t / fl(a_t + x)),  a_t = fl(vbar_t + eps_b),
 *              (q_t = 0 where a_t is not positive and finite), and
 *                  c = the smallest x among the non-negative floats and +inf
 *                      with E(x) <= min(B, P) * 2^32.
 *              Every q_t is non-increasing in x (IEEE rounding is monotone),
 *              so E is too and c is unique; E(+inf) = 0, so c exists.  The
 *              terms are integers (fixed point, 2^-32 parameters), so the sum
 *              is exact in any order.  A tensor with a larger vbar gets a
 *              larger share: the expected share of tensor t is s_t a_t /
 *              (a_t + c), the allocation "according to likelihood of
 *              staleness" of the future-work section.
 *   draws      u_t = word (t mod 4) of Philox4x32-10 at counter
 *              (2^31 + t div 4, client + 2^31 * stream, n, n >> 32), top 24
 *              bits, n = the client's count of earlier pushes (stream 0) or
 *              fetches (stream 1); the first counter word never meets the
 *              per-parameter draws (p div 4 < 2^29) or the per-message draw
 *              (2^32 - 1) for t < 2^31 - 4.
 *   unsent     a tensor that is not transmitted is not updated (the same
 *              reading as the per-parameter path).
 */

/* vbar_t for every tensor: the exact mean over the tensor, rounded once. */
void ora_tensor_means(int32_t T, const int64_t *sizes, const REAL *v, float *vbar)
{
    int64_t off = 0;
    for (int32_t t = 0; t < T; t++) {
        ora_exact_sum s;
        ora_sum_clear(&s);
        for (int64_t p = off; p < off + sizes[t]; p++)
            ora_sum_add(&s, (double)v[p]);
        vbar[t] = ora_sum_mean(&s, sizes[t]);
        off += sizes[t];
    }
}

/* floor(size * q * 2^32) for q = fl(a / fl(a + x)), exactly, in integers. */
static int64_t ora_budget_term(int64_t size, float vbar, float eps_b, float x)
{
    float a = vbar + eps_b;
    if (!(a > 0.0f) || isinf(a))
        return 0;
    float d = a + x;
    float q = a / d;
    if (q == 0.0f)
        return 0;
    int e;
    float m = frexpf(q, &e);                   /* q = m 2^e, 1/2 <= m < 1 */
    int64_t M = (int64_t)ldexpf(m, 24);        /* integer, exact: at most 24 bits */
    int64_t prod = size * M;                   /* < 2^31 * 2^24 */
    int shift = e - 24 + 32;                   /* size * q * 2^32 = prod * 2^shift */
    if (shift >= 0)
        return prod << shift;                  /* q <= 1, so at most size * 2^32 */
    if (shift <= -63)
        return 0;
    return prod >> (-shift);
}

/* E(x): expected parameters sent at threshold x, in units of 2^-32. */
int64_t ora_budget_expected(int32_t T, const int64_t *sizes, const float *vbar, float eps_b,
                            float x)
{
    int64_t e = 0;
    for (int32_t t = 0; t < T; t++)
        e += ora_budget_term(sizes[t], vbar[t], eps_b, x);
    return e;
}

static float ora_float_of_bits(uint32_t bits)
{
    float f;
    memcpy(&f, &bits, sizeof f);
    return f;
}

/* The budget threshold c (above): bisection over the bit patterns of the
 * non-negative floats, which are ordered like the values they encode. */
float ora_budget_c(int32_t T, const int64_t *sizes, const float *vbar, float eps_b,
                   int64_t budget)
{
    int64_t S = 0;
    for (int32_t t = 0; t < T; t++)
        S += sizes[t];
    int64_t B = budget < 0 ? 0 : (budget > S ? S : budget);
    int64_t limit = B * ((int64_t)1 << 32);
    if (ora_budget_expected(T, sizes, vbar, eps_b, 0.0f) <= limit)
        return 0.0f;
    uint32_t lo = 0, hi = 0x7F800000u;        /* E(lo) > limit >= E(hi) = E(+inf) */
    while (hi - lo > 1) {
        uint32_t mid = lo + (hi - lo) / 2;
        if (ora_budget_expected(T, sizes, vbar, eps_b, ora_float_of_bits(mid)) <= limit)
            hi = mid;
        else
            lo = mid;
    }
    return ora_float_of_bits(hi);
}

uint32_t ora_draw_tensor(uint64_t seed, uint32_t stream, uint32_t client, uint64_t n, int32_t t)
{
    uint32_t ctr[4] = {0x80000000u + ((uint32_t)t >> 2), client | (stream << 31), (uint32_t)n,
                       (uint32_t)(n >> 32)};
    uint32_t key[2] = {(uint32_t)seed, (uint32_t)(seed >> 32)};
    uint32_t out[4];
    ora_philox4x32_10(ctr, key, out);
    return out[t & 3] >> 8;
}

/* The per-tensor decisions at threshold c; returns the parameters transmitted. */
int64_t ora_tensor_select(int32_t T, const int64_t *sizes, const float *vbar, float c,
                          float eps_b, uint64_t seed, uint32_t stream, uint32_t client,
                          uint64_t n, uint8_t *sent)
{
    int64_t m = 0;
    for (int32_t t = 0; t < T; t++) {
        uint32_t u = ora_draw_tensor(seed, stream, client, n, t);
        sent[t] = (uint8_t)ora_decide(u, vbar[t], c, eps_b);
        if (sent[t])
            m += sizes[t];
    }
    return m;
}

/* A per-tensor push: every parameter of a transmitted tensor receives g[p]. */
void ora_apply_tensors(int variant, int32_t T, const int64_t *sizes, const uint8_t *sent,
                       REAL *theta, REAL *n, REAL *b, REAL *v, const float *g, REAL coef,
                       REAL gamma, REAL beta, REAL eps)
{
    int64_t off = 0;
    for (int32_t t = 0; t < T; t++) {
        if (sent[t])
            for (int64_t p = off; p < off + sizes[t]; p++)
                ora_update_one(variant, &theta[p], &n[p], &b[p], &v[p], (REAL)g[p], coef,
                               gamma, beta, eps);
        off += sizes[t];
    }
}
