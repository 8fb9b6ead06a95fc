/*
 * adpsgd_oracle.c -- plain, slow CPU oracle for the data-parallel hot path of
 * ADPSGD (Jiang & Agrawal, "Adaptive Periodic Averaging", arXiv 2007.06134).
 *
 * TEST INFRASTRUCTURE ONLY.  Only the tests, the smoke check and the CPU
 * baseline leg of the benchmark may load this file's library.  The product
 * path (the CUDA library) shares no code, header, table or constant with it.
 *
 * What it computes, each piece written in the most literal form:
 *   - Philox4x32-10 (Salmon, Moraes, Dror, Shaw, SC'11), the counter-based
 *     generator that stands in for mini-batch sampling noise (Sec. II-A, Eq. eg).
 *   - Box-Muller (Box & Muller 1958) on top of it, with a natural log (atanh
 *     series) and a sine/cosine of 2*pi*u (Taylor series after an exact
 *     quarter-turn reduction) built only from correctly rounded IEEE
 *     operations (+ - * / sqrt fma), so that any IEEE machine gets the same bits.
 *   - The local step of Algorithm 1 (update line) and Algorithm 2 (update line)
 *     on the surrogate objective f(x) = 1/2 sum_j h_j (x_j - c_j)^2, with SGD
 *     momentum and weight decay in the PyTorch 1.0 convention the experiments
 *     used (Sec. IV-A gives the momentum, 0.9, and nothing else about it).
 *   - Parameter averaging (Algorithm 2, averaging line; Eq. alg1's A_n) and the
 *     inter-replica variance of Sec. II-B (definition of Var[W_k]) and S_k of
 *     Algorithm 2, plus the surrogate loss at the average.
 *   - The period rule of Algorithm 2 (cnt, p, C_2; sampling phase k < K_s;
 *     +1 / -1 at 0.7 and 1.3) and Algorithm 1 as the constant-period case.
 *   - The bytes a ring allreduce would put on the wire per schedule.
 *   - The same run on all host cores (OpenMP over fixed column chunks, the
 *     fp64 partial sums added in chunk order), for full-size comparisons.
 *
 * Precision.  Parameters and momentum buffers are fp32 (the experiments ran
 * PyTorch 1.0 defaults); every fp32 operation below is separately rounded
 * (build with -ffp-contract=off, no fast-math).  Reductions (variance, loss)
 * are the plain definition evaluated in fp64.
 *
 * Readings of the paper taken here (the paper is silent or ambiguous):
 *   R1 momentum: v = mu*v + g; x = x - gamma*v; weight decay added to g.
 *   R2 momentum buffers are never averaged (Algorithm 2 averages w only).
 *   R3 the replica mean is formed as x_0 + (sum_{i>=1} (x_i - x_0)) / n in
 *      fp32 -- equal to (1/n) sum_i x_i in exact arithmetic -- so that the
 *      variance right after averaging is exactly zero (Sec. III-B) and n = 1 is
 *      exactly the identity.
 *   R4 S_k = D / n with D = sum_i ||x_i - xbar||^2 (Sec. II-B definition of Var).
 *   R5 RunningAverage = cumulative arithmetic mean of S_k / gamma_k.
 *   R6 p is clamped to [p_min, p_max] (p_max = 0: no upper bound).
 *   R7 the constant-period schedule syncs when cnt reaches p (as Algorithm 2
 *      with adaptation off); Algorithm 1's literal "k mod p == 0" is a flag.
 *   R8 optional warm-up: the first K_w iterations sync every iteration and are
 *      not sampled into C_2 (Sec. IV-B).
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

/* ------------------------------------------------------------------------ */
/* Philox4x32-10.  State of four 32-bit words, key of two.  One round:       */
/* multiply words 0 and 2 by the two round multipliers, keep both halves of  */
/* each 64-bit product, and xor the high halves with the other two words and */
/* the key.  Between rounds the key is bumped by the two Weyl constants.     */
/* ------------------------------------------------------------------------ */
#define PHILOX_M0 0xD2511F53u
#define PHILOX_M1 0xCD9E8D57u
#define PHILOX_W0 0x9E3779B9u
#define PHILOX_W1 0xBB67AE85u

static void philox_one_round(uint32_t c[4], const uint32_t key[2])
{
    uint64_t prod0 = (uint64_t)PHILOX_M0 * (uint64_t)c[0];
    uint64_t prod1 = (uint64_t)PHILOX_M1 * (uint64_t)c[2];
    uint32_t hi0 = (uint32_t)(prod0 >> 32), lo0 = (uint32_t)prod0;
    uint32_t hi1 = (uint32_t)(prod1 >> 32), lo1 = (uint32_t)prod1;
    uint32_t out0 = hi1 ^ c[1] ^ key[0];
    uint32_t out1 = lo1;
    uint32_t out2 = hi0 ^ c[3] ^ key[1];
    uint32_t out3 = lo0;
    c[0] = out0; c[1] = out1; c[2] = out2; c[3] = out3;
}

void orc_philox4x32_10(const uint32_t ctr[4], const uint32_t key[2], uint32_t out[4])
{
    uint32_t c[4] = {ctr[0], ctr[1], ctr[2], ctr[3]};
    uint32_t k[2] = {key[0], key[1]};
    for (int round = 0; round < 10; ++round) {
        if (round > 0) {
            k[0] += PHILOX_W0;
            k[1] += PHILOX_W1;
        }
        philox_one_round(c, k);
    }
    for (int w = 0; w < 4; ++w) out[w] = c[w];
}

/* The counter layout of the noise stream: element j of replica i at step k  */
/* takes word (j mod 4) of Philox(counter = (j div 4, i, k, tag),            */
/* key = (seed low 32 bits, seed high 32 bits)).                             */
static void noise_words(uint64_t seed, uint32_t tag, uint32_t i, uint32_t k, uint64_t q, uint32_t w[4])
{
    uint32_t ctr[4] = {(uint32_t)q, i, k, tag};
    uint32_t key[2] = {(uint32_t)(seed & 0xffffffffu), (uint32_t)(seed >> 32)};
    orc_philox4x32_10(ctr, key, w);
}

void orc_philox_words(uint64_t seed, uint32_t tag, uint32_t i, uint32_t k, int64_t q0, int64_t nq, uint32_t* out)
{
    for (int64_t t = 0; t < nq; ++t) noise_words(seed, tag, i, k, (uint64_t)(q0 + t), out + 4 * t);
}

/* ------------------------------------------------------------------------ */
/* Uniforms from a 32-bit word, 23 bits each, exact in fp32.                 */
/*   open at 0:  u = 1 - (w >> 9) * 2^-23   in [2^-23, 1]   (feeds the log)  */
/*   half-open:  u = (w >> 9) * 2^-23       in [0, 1 - 2^-23] (the angle)    */
/* ------------------------------------------------------------------------ */
static float uniform_open0(uint32_t w) { return 1.0f - (float)(w >> 9) * 0x1p-23f; }
static float uniform_half(uint32_t w) { return (float)(w >> 9) * 0x1p-23f; }

/* ------------------------------------------------------------------------ */
/* Natural log for a positive normal fp32 u.                                 */
/* u = 2^e * m with m in [sqrt(1/2), sqrt(2)); ln u = e ln2 + ln m, and      */
/* ln m = 2 atanh(s) = 2 (s + s^3/3 + s^5/5 + ...) with s = (m-1)/(m+1),     */
/* |s| <= 0.1716.  Terms up to s^11/11 (the next one is below 1e-12).         */
/* ln2 is split as LN2_HI (15 significant bits, so e*LN2_HI is exact for     */
/* |e| < 2^9) plus LN2_LO (Cody & Waite).                                    */
/* ------------------------------------------------------------------------ */
static const float ORC_SQRT2 = 1.41421356237309504880f;
static const float ORC_LN2_HI = 0.693145751953125f;        /* 0x3F317200 */
static const float ORC_LN2_LO = 1.42860682030941723212e-6f; /* ln2 - LN2_HI */

float orc_ln(float u)
{
    int e;
    float m = frexpf(u, &e);      /* u = m * 2^e, m in [0.5, 1) */
    m = 2.0f * m;                 /* m in [1, 2) */
    e = e - 1;
    if (m >= ORC_SQRT2) {         /* move m into [sqrt(1/2), sqrt(2)) */
        m = 0.5f * m;
        e = e + 1;
    }
    float s = (m - 1.0f) / (m + 1.0f);
    float s2 = s * s;
    float poly = 1.0f / 11.0f;
    poly = fmaf(poly, s2, 1.0f / 9.0f);
    poly = fmaf(poly, s2, 1.0f / 7.0f);
    poly = fmaf(poly, s2, 1.0f / 5.0f);
    poly = fmaf(poly, s2, 1.0f / 3.0f);
    float tail = s * (s2 * poly);       /* s^3/3 + s^5/5 + ... */
    float atanh_s = s + tail;
    float ln_m = 2.0f * atanh_s;
    float ef = (float)e;
    return ef * ORC_LN2_HI + (ef * ORC_LN2_LO + ln_m);
}

/* ------------------------------------------------------------------------ */
/* sin and cos of 2*pi*u for u in [0, 1).                                    */
/* t = 4u (exact) = q + r with q = nearest integer (ties to even) and        */
/* r in [-1/2, 1/2] (exact).  Then 2*pi*u = q*pi/2 + r*pi/2 and the quarter  */
/* turn q only permutes and negates sin and cos of phi = r*pi/2,             */
/* |phi| <= pi/4.  Taylor series in r:                                       */
/*   sin(phi) = sum_k (-1)^k (pi/2)^(2k+1) r^(2k+1) / (2k+1)!   up to r^9    */
/*   cos(phi) = sum_k (-1)^k (pi/2)^(2k)   r^(2k)   / (2k)!     up to r^10   */
/* The first dropped terms are below 2e-9 and 2e-10.                          */
/* ------------------------------------------------------------------------ */
/* (pi/2)^k / k!, with the sign of the series, k = 1, 3, 5, 7, 9 */
static const float ORC_S1 = 1.57079632679489661923f;
static const float ORC_S3 = -0.645964097506246253656f;
static const float ORC_S5 = 0.0796926262461670451205f;
static const float ORC_S7 = -0.00468175413531868810068f;
static const float ORC_S9 = 0.000160441184787359821873f;
/* k = 2, 4, 6, 8, 10 */
static const float ORC_C2 = -1.23370055013616982735f;
static const float ORC_C4 = 0.253669507901048013637f;
static const float ORC_C6 = -0.0208634807633529608730f;
static const float ORC_C8 = 0.000919260274839426580242f;
static const float ORC_C10 = -0.0000252020423730606054811f;

void orc_sincos_turn(float u, float* sin_out, float* cos_out)
{
    float t = 4.0f * u;
    float q = nearbyintf(t);      /* default rounding mode: ties to even */
    float r = t - q;
    float r2 = r * r;
    float ps = ORC_S9;
    ps = fmaf(ps, r2, ORC_S7);
    ps = fmaf(ps, r2, ORC_S5);
    ps = fmaf(ps, r2, ORC_S3);
    ps = fmaf(ps, r2, ORC_S1);
    float sin_phi = ps * r;
    float pc = ORC_C10;
    pc = fmaf(pc, r2, ORC_C8);
    pc = fmaf(pc, r2, ORC_C6);
    pc = fmaf(pc, r2, ORC_C4);
    pc = fmaf(pc, r2, ORC_C2);
    float cos_phi = fmaf(pc, r2, 1.0f);
    int quarter = ((int)q) & 3;
    float s, c;
    switch (quarter) {
    case 0: s = sin_phi;  c = cos_phi;  break;
    case 1: s = cos_phi;  c = -sin_phi; break;
    case 2: s = -sin_phi; c = -cos_phi; break;
    default: s = -cos_phi; c = sin_phi; break;
    }
    *sin_out = s;
    *cos_out = c;
}

/* Box-Muller: radius sqrt(-2 ln u1), angle 2*pi*u2; z0 = r cos, z1 = r sin. */
static void box_muller(uint32_t w_radius, uint32_t w_angle, float* z0, float* z1)
{
    float u1 = uniform_open0(w_radius);
    float u2 = uniform_half(w_angle);
    float radius = sqrtf(-2.0f * orc_ln(u1));
    float s, c;
    orc_sincos_turn(u2, &s, &c);
    *z0 = radius * c;
    *z1 = radius * s;
}

/* Box-Muller on raw words (exposed so that tests can feed chosen words). */
void orc_box_muller_words(uint32_t w_radius, uint32_t w_angle, float* z0, float* z1)
{
    box_muller(w_radius, w_angle, z0, z1);
}

/* The same over arrays of word pairs (for exhaustive comparisons). */
void orc_box_muller_array(const uint32_t* w_radius, const uint32_t* w_angle, int64_t m, float* z0, float* z1)
{
    for (int64_t t = 0; t < m; ++t) box_muller(w_radius[t], w_angle[t], &z0[t], &z1[t]);
}

/* The four normals of one Philox block: words (0,1) -> elements 4q+0, 4q+1, */
/* words (2,3) -> elements 4q+2, 4q+3.                                       */
static void normals_of_block(uint64_t seed, uint32_t tag, uint32_t i, uint32_t k, uint64_t q, float z[4])
{
    uint32_t w[4];
    noise_words(seed, tag, i, k, q, w);
    box_muller(w[0], w[1], &z[0], &z[1]);
    box_muller(w[2], w[3], &z[2], &z[3]);
}

/* Gaussian noise z[i, j] for step k, elements j0 .. j0+m-1 of replica i. */
void orc_normals(uint64_t seed, uint32_t tag, uint32_t i, uint32_t k, int64_t j0, int64_t m, float* out)
{
    for (int64_t t = 0; t < m; ++t) {
        int64_t j = j0 + t;
        float z[4];
        normals_of_block(seed, tag, i, k, (uint64_t)(j / 4), z);
        out[t] = z[j % 4];
    }
}

void orc_ln_array(const float* u, float* out, int64_t m)
{
    for (int64_t t = 0; t < m; ++t) out[t] = orc_ln(u[t]);
}

void orc_sincos_array(const float* u, float* s, float* c, int64_t m)
{
    for (int64_t t = 0; t < m; ++t) orc_sincos_turn(u[t], &s[t], &c[t]);
}

/* fp32 -> bf16, round to nearest even (finite inputs). */
static uint16_t to_bf16(float f)
{
    uint32_t b;
    memcpy(&b, &f, 4);
    uint32_t lsb = (b >> 16) & 1u;
    b = b + 0x7FFFu + lsb;
    return (uint16_t)(b >> 16);
}

static float from_bf16(uint16_t h)
{
    uint32_t b = (uint32_t)h << 16;
    float f;
    memcpy(&f, &b, 4);
    return f;
}

void orc_to_bf16_array(const float* in, uint16_t* out, int64_t m)
{
    for (int64_t t = 0; t < m; ++t) out[t] = to_bf16(in[t]);
}

/* The pre-materialised bf16 noise tensor [n, P]: the step-0 normals of the  */
/* stream with tag 1, rounded to bf16.                                       */
void orc_noise_bf16(uint64_t seed, int32_t n, int64_t P, uint16_t* out)
{
    /* rows are independent: one host thread per row (OpenMP) */
    #pragma omp parallel for schedule(static)
    for (int32_t i = 0; i < n; ++i)
        for (int64_t j = 0; j < P; ++j) {
            float z[4];
            normals_of_block(seed, 1u, (uint32_t)i, 0u, (uint64_t)(j / 4), z);
            out[(int64_t)i * P + j] = to_bf16(z[j % 4]);
        }
}

/* ------------------------------------------------------------------------ */
/* Local step (Algorithm 1 / Algorithm 2, the local update), for every     */
/* replica i and columns j in [j0, j1).                                      */
/* Stochastic gradient of the surrogate: g = h_j (x - c_j) + sigma * z.      */
/* Reading R1: g += wd * x (only when wd != 0); v = mu * v + g;              */
/* x = x - gamma * v.  Each operation is one fp32 rounding.                  */
/* noise_bf16 == NULL: z from the Philox stream (tag 0) at step k;           */
/* otherwise z = noise_bf16[i, j] (the same tensor every step).              */
/* ------------------------------------------------------------------------ */
void orc_local_step(int32_t n, int64_t P, int64_t j0, int64_t j1, float* x, float* v,
                    const float* h, const float* c, const uint16_t* noise_bf16, uint64_t seed,
                    int64_t k, float gamma, float mu, float wd, float sigma)
{
    for (int32_t i = 0; i < n; ++i) {
        float* xi = x + (int64_t)i * P;
        float* vi = v + (int64_t)i * P;
        float zb[4] = {0.0f, 0.0f, 0.0f, 0.0f};
        int64_t block = -1;  /* the Philox block whose four normals zb holds */
        for (int64_t j = j0; j < j1; ++j) {
            float z;
            if (noise_bf16 != NULL) {
                z = from_bf16(noise_bf16[(int64_t)i * P + j]);
            } else {
                if (j / 4 != block) {
                    block = j / 4;
                    normals_of_block(seed, 0u, (uint32_t)i, (uint32_t)k, (uint64_t)block, zb);
                }
                z = zb[j % 4];
            }
            float diff = xi[j] - c[j];
            float g = h[j] * diff;
            float noise = sigma * z;
            g = g + noise;
            if (wd != 0.0f) {
                float decay = wd * xi[j];
                g = g + decay;
            }
            float mv = mu * vi[j];
            float vnew = mv + g;
            float step = gamma * vnew;
            vi[j] = vnew;
            xi[j] = xi[j] - step;
        }
    }
}

/* ------------------------------------------------------------------------ */
/* Averaging and variance (Algorithm 2, averaging and S_k lines; Sec. II-B   */
/* definition of Var[W_k]) for columns [j0, j1).                             */
/* xbar_j (fp32, reading R3) is written back to every replica.               */
/* *D    += sum_j sum_i (x_ij - xbar_j)^2   in fp64 (before the write-back)  */
/* *loss += 1/2 sum_j h_j (xbar_j - c_j)^2  in fp64 (if loss != NULL)        */
/* ------------------------------------------------------------------------ */
void orc_average_variance(int32_t n, int64_t P, int64_t j0, int64_t j1, float* x,
                          const float* h, const float* c, double* D, double* loss)
{
    double dsum = 0.0, lsum = 0.0;
    for (int64_t j = j0; j < j1; ++j) {
        float base = x[j];
        float acc = 0.0f;
        for (int32_t i = 1; i < n; ++i) acc = acc + (x[(int64_t)i * P + j] - base);
        float xbar = base + acc / (float)n;
        for (int32_t i = 0; i < n; ++i) {
            double dev = (double)x[(int64_t)i * P + j] - (double)xbar;
            dsum += dev * dev;
        }
        if (loss != NULL) {
            double r = (double)xbar - (double)c[j];
            lsum += 0.5 * (double)h[j] * r * r;
        }
        for (int32_t i = 0; i < n; ++i) x[(int64_t)i * P + j] = xbar;
    }
    *D += dsum;
    if (loss != NULL) *loss += lsum;
}

/* Variance only (no write-back) of columns [j0, j1), for per-iteration diagnostics: D as above. */
double orc_variance_cols(int32_t n, int64_t P, int64_t j0, int64_t j1, const float* x)
{
    double dsum = 0.0;
    for (int64_t j = j0; j < j1; ++j) {
        float base = x[j];
        float acc = 0.0f;
        for (int32_t i = 1; i < n; ++i) acc = acc + (x[(int64_t)i * P + j] - base);
        float xbar = base + acc / (float)n;
        for (int32_t i = 0; i < n; ++i) {
            double dev = (double)x[(int64_t)i * P + j] - (double)xbar;
            dsum += dev * dev;
        }
    }
    return dsum;
}

double orc_variance(int32_t n, int64_t P, const float* x) { return orc_variance_cols(n, P, 0, P, x); }

/* ------------------------------------------------------------------------ */
/* Schedules.                                                                */
/* ------------------------------------------------------------------------ */
typedef struct {
    int32_t kind;          /* 0 constant period (Algorithm 1), 1 adaptive (Algorithm 2),
                              2 piecewise-constant period (the strategies of Sec. III-A and the
                              decreasing period of Sec. V-B) */
    int32_t p_init;        /* constant p, or p_init */
    int64_t K;             /* iterations */
    int64_t K_s;           /* sampling phase: syncs at k < K_s sample C_2 */
    int64_t K_w;           /* warm-up iterations with p = 1 (R8) */
    double lo, hi;         /* 0.7 and 1.3 */
    int32_t p_min, p_max;  /* clamp of p (R6); p_max = 0: none */
    double lr0;            /* gamma at k = 0 */
    double lr_factor;      /* gamma multiplied by this at each milestone */
    int32_t n_milestones;
    int32_t literal_phase; /* constant period only: sync when k mod p == 0 */
    const int64_t* milestones; /* gamma changes from iteration milestones[t] on */
    int32_t n_period_changes;  /* kind 2: p = period_values[t] from iteration period_change_k[t] on */
    int32_t pad;
    const int64_t* period_change_k;
    const int32_t* period_values;
    int32_t lr_warmup_steps;   /* step-size warm-up (Sec. IV-C): gamma = lr0 * (s + 1) on stair s,   */
    int32_t pad2;              /* s = min(k div lr_warmup_len, lr_warmup_steps - 1); 0: no warm-up */
    int64_t lr_warmup_len;
} orc_schedule;

typedef struct {
    int32_t cnt;  /* iterations since the last sync */
    int32_t p;    /* current period */
    double C2;    /* sampled constant */
    int64_t m;    /* number of samples in C2 */
} orc_state;

/* Step size of iteration k: lr0 (times the warm-up stair multiple), times */
/* lr_factor once per milestone <= k, in fp64, then rounded once to fp32.  */
float orc_gamma(const orc_schedule* s, int64_t k)
{
    double g = s->lr0;
    if (s->lr_warmup_steps > 0) {
        int64_t stair = k / s->lr_warmup_len;
        if (stair > s->lr_warmup_steps - 1) stair = s->lr_warmup_steps - 1;
        g = g * (double)(stair + 1);
    }
    for (int32_t t = 0; t < s->n_milestones; ++t)
        if (k >= s->milestones[t]) g = g * s->lr_factor;
    return (float)g;
}

/* Period in force at iteration k for kind 2: p_init, replaced by period_values[t] from   */
/* iteration period_change_k[t] on.                                                       */
static int32_t period_at(const orc_schedule* s, int64_t k)
{
    int32_t p = s->p_init;
    for (int32_t t = 0; t < s->n_period_changes; ++t)
        if (k >= s->period_change_k[t]) p = s->period_values[t];
    return p;
}

/* Phase codes recorded per sync. */
enum { ORC_PHASE_CONSTANT = 0, ORC_PHASE_WARMUP = 1, ORC_PHASE_SAMPLING = 2, ORC_PHASE_ADAPTING = 3 };

/* The period rule of Algorithm 2 after a sync at iteration k with variance */
/* S and step size gamma.  Returns the phase code.                          */
int32_t orc_on_sync(const orc_schedule* s, orc_state* st, int64_t k, double S, double gamma)
{
    if (k < s->K_w) return ORC_PHASE_WARMUP;
    if (s->kind == 0 || s->kind == 2) return ORC_PHASE_CONSTANT;
    if (k < s->K_s) {
        st->m = st->m + 1;
        st->C2 = st->C2 + (S / gamma - st->C2) / (double)st->m;
        return ORC_PHASE_SAMPLING;
    }
    double target = gamma * st->C2;
    if (S < s->lo * target) {
        st->p = st->p + 1;
    } else if (S > s->hi * target) {
        st->p = st->p - 1;
    }
    if (st->p < s->p_min) st->p = s->p_min;
    if (s->p_max > 0 && st->p > s->p_max) st->p = s->p_max;
    return ORC_PHASE_ADAPTING;
}

/* Does the iteration that just finished (index k) end with a sync?        */
/* Advances cnt as Algorithm 2 does.                                        */
static int sync_now(const orc_schedule* s, orc_state* st, int64_t k)
{
    if (k < s->K_w) {
        st->cnt = 0;
        return 1;
    }
    if (s->kind == 2) st->p = period_at(s, k);
    if (s->kind == 0 && s->literal_phase) return (k % st->p) == 0;
    st->cnt = st->cnt + 1;
    if (st->cnt >= st->p) {
        st->cnt = 0;
        return 1;
    }
    return 0;
}

typedef struct {
    int64_t* k;      /* iteration of the sync */
    int32_t* p;      /* period after the rule ran */
    double* S;       /* D / n */
    double* C2;      /* C_2 after the rule ran */
    double* loss;    /* surrogate loss at the average */
    int32_t* phase;  /* phase code */
    int64_t cap;     /* capacity of the arrays */
    double* var;     /* optional: var[k] = Var[W_k] (Sec. II-B) at the start of iteration k */
    int64_t var_cap; /* entries of var */
} orc_trace;

/* Initial scheduler state. */
void orc_state_init(const orc_schedule* s, orc_state* st)
{
    st->cnt = 0;
    st->p = s->p_init;
    st->C2 = 0.0;
    st->m = 0;
}

/* Run iterations k in [k_begin, k_end) of the schedule from state st on the */
/* [n, P] arrays.  Returns the number of syncs; records up to trace->cap.   */
int64_t orc_run(int32_t n, int64_t P, float* x, float* v, const float* h, const float* c,
                const uint16_t* noise_bf16, uint64_t seed, float mu, float wd, float sigma,
                const orc_schedule* s, orc_state* st, int64_t k_begin, int64_t k_end, orc_trace* tr)
{
    int64_t syncs = 0;
    for (int64_t k = k_begin; k < k_end; ++k) {
        float gamma = orc_gamma(s, k);
        if (tr != NULL && tr->var != NULL && k < tr->var_cap) tr->var[k] = orc_variance(n, P, x) / (double)n;
        orc_local_step(n, P, 0, P, x, v, h, c, noise_bf16, seed, k, gamma, mu, wd, sigma);
        if (!sync_now(s, st, k)) continue;
        double D = 0.0, loss = 0.0;
        orc_average_variance(n, P, 0, P, x, h, c, &D, &loss);
        double S = D / (double)n;
        int32_t phase = orc_on_sync(s, st, k, S, (double)gamma);
        if (tr != NULL && syncs < tr->cap) {
            tr->k[syncs] = k;
            tr->p[syncs] = st->p;
            tr->S[syncs] = S;
            tr->C2[syncs] = st->C2;
            tr->loss[syncs] = loss;
            tr->phase[syncs] = phase;
        }
        syncs = syncs + 1;
    }
    return syncs;
}

/* ------------------------------------------------------------------------ */
/* The same run on several host threads (OpenMP).  The columns are cut into  */
/* fixed chunks of `chunk` columns, a multiple of 4 so that no Philox block  */
/* is split; each thread runs the per-element code above on whole chunks.   */
/* The fp64 partial sums of D and the loss (and of the per-iteration         */
/* variance) are kept per chunk and added in chunk order, so the result does */
/* not depend on the thread count.  x, v, the sync iterations, the periods   */
/* and the phases equal orc_run's bit for bit; D and the loss differ from    */
/* orc_run's only in the order of their fp64 additions.                      */
/* Returns the number of syncs, or -1 if chunk is not a positive multiple    */
/* of 4 or the partial sums cannot be allocated.                             */
/* ------------------------------------------------------------------------ */
int64_t orc_run_chunked(int32_t threads, int64_t chunk, int32_t n, int64_t P, float* x, float* v,
                        const float* h, const float* c, const uint16_t* noise_bf16, uint64_t seed,
                        float mu, float wd, float sigma, const orc_schedule* s, orc_state* st,
                        int64_t k_begin, int64_t k_end, orc_trace* tr)
{
    if (chunk <= 0 || chunk % 4 != 0) return -1;
    const int64_t nchunks = (P + chunk - 1) / chunk;
    double* part = (double*)calloc((size_t)(2 * nchunks + 1), sizeof(double));
    if (part == NULL) return -1;
    double* partD = part;
    double* partL = part + nchunks;
    if (threads < 1) threads = 1;
    int64_t syncs = 0;
    for (int64_t k = k_begin; k < k_end; ++k) {
        float gamma = orc_gamma(s, k);
        if (tr != NULL && tr->var != NULL && k < tr->var_cap) {
            #pragma omp parallel for num_threads(threads) schedule(static)
            for (int64_t ch = 0; ch < nchunks; ++ch) {
                const int64_t j1 = (ch + 1) * chunk < P ? (ch + 1) * chunk : P;
                partD[ch] = orc_variance_cols(n, P, ch * chunk, j1, x);
            }
            double D = 0.0;
            for (int64_t ch = 0; ch < nchunks; ++ch) D += partD[ch];
            tr->var[k] = D / (double)n;
        }
        #pragma omp parallel for num_threads(threads) schedule(static)
        for (int64_t ch = 0; ch < nchunks; ++ch) {
            const int64_t j1 = (ch + 1) * chunk < P ? (ch + 1) * chunk : P;
            orc_local_step(n, P, ch * chunk, j1, x, v, h, c, noise_bf16, seed, k, gamma, mu, wd, sigma);
        }
        if (!sync_now(s, st, k)) continue;
        #pragma omp parallel for num_threads(threads) schedule(static)
        for (int64_t ch = 0; ch < nchunks; ++ch) {
            const int64_t j1 = (ch + 1) * chunk < P ? (ch + 1) * chunk : P;
            partD[ch] = 0.0;
            partL[ch] = 0.0;
            orc_average_variance(n, P, ch * chunk, j1, x, h, c, &partD[ch], &partL[ch]);
        }
        double D = 0.0, loss = 0.0;
        for (int64_t ch = 0; ch < nchunks; ++ch) {
            D += partD[ch];
            loss += partL[ch];
        }
        double S = D / (double)n;
        int32_t phase = orc_on_sync(s, st, k, S, (double)gamma);
        if (tr != NULL && syncs < tr->cap) {
            tr->k[syncs] = k;
            tr->p[syncs] = st->p;
            tr->S[syncs] = S;
            tr->C2[syncs] = st->C2;
            tr->loss[syncs] = loss;
            tr->phase[syncs] = phase;
        }
        syncs = syncs + 1;
    }
    free(part);
    return syncs;
}

/* Schedule only: the sync iterations and periods when every sync reports   */
/* the variance S_of_sync[t] (scripted), without any arithmetic on arrays.  */
int64_t orc_schedule_only(const orc_schedule* s, const double* S_of_sync, int64_t n_scripted,
                          int64_t* k_out, int32_t* p_out, int64_t cap)
{
    orc_state st;
    orc_state_init(s, &st);
    int64_t syncs = 0;
    for (int64_t k = 0; k < s->K; ++k) {
        if (!sync_now(s, &st, k)) continue;
        double S = syncs < n_scripted ? S_of_sync[syncs] : 0.0;
        orc_on_sync(s, &st, k, S, (double)orc_gamma(s, k));
        if (syncs < cap) {
            k_out[syncs] = k;
            p_out[syncs] = st.p;
        }
        syncs = syncs + 1;
    }
    return syncs;
}

/* ------------------------------------------------------------------------ */
/* Wire accounting.  A ring allreduce of b bytes moves 2 (n-1)/n * b bytes  */
/* in and out of every node (reduce-scatter then all-gather).  Each sync   */
/* of Algorithm 2 allreduces P fp32 parameters and one fp32 S_k.           */
/* Full-communication SGD allreduces P fp32 gradients every iteration.     */
/* ------------------------------------------------------------------------ */
void orc_wire_bytes(int32_t n, int64_t P, int64_t rounds, int32_t with_scalar,
                    double* per_node, double* total)
{
    double ring = 2.0 * (double)(n - 1) / (double)n;
    double per_round = ring * 4.0 * (double)P;
    if (with_scalar) per_round += ring * 4.0;
    *per_node = per_round * (double)rounds;
    *total = *per_node * (double)n;
}
