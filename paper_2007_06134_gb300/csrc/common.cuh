// common.cuh -- device arithmetic shared by the kernels of this library: the SGD update of one
// element, the per-column mean and squared deviations, and a fixed-order block sum.  Compiled
// with -fmad=false: every operation written here is one IEEE rounding.
#pragma once

#include <cstdint>

namespace adpsgd {

constexpr int kThreads = 256;

// g = h (x - c) + sigma z [+ wd x];  v = mu v + g;  x = x - gamma v  (one rounding each).
template <bool WD>
__device__ __forceinline__ void sgd_update(float& x, float& v, float h, float c, float z,
                                           float gamma, float mu, float wd, float sigma)
{
    const float diff = x - c;
    float g = h * diff;
    const float noise = sigma * z;
    g = g + noise;
    if (WD) {
        const float decay = wd * x;
        g = g + decay;
    }
    const float mv = mu * v;
    const float vnew = mv + g;
    const float step = gamma * vnew;
    v = vnew;
    x = x - step;
}

__device__ __forceinline__ float bf16_bits_to_float(uint32_t bits16) { return __uint_as_float(bits16 << 16); }

// Fixed-order block sum over a block of THREADS threads (shared: THREADS / 32 doubles); the
// result is valid in thread 0.
template <int THREADS = kThreads>
__device__ __forceinline__ double block_sum(double v, double* shared)
{
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) v += __shfl_down_sync(0xFFFFFFFFu, v, off);
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    if (lane == 0) shared[warp] = v;
    __syncthreads();
    double total = 0.0;
    if (threadIdx.x == 0)
        for (int w = 0; w < THREADS / 32; ++w) total += shared[w];
    __syncthreads();
    return total;
}

// The mean's offset acc / n (n > 0) in IEEE fp32.  An exact zero numerator (identical replicas, or
// deviations that cancel) is its own quotient, sign included, so it skips the division, whose
// handling of a zero operand measured about twice the instructions of the whole averaging on
// identical replicas.
__device__ __forceinline__ float mean_offset(float acc, float nf) { return acc == 0.0f ? acc : __fdiv_rn(acc, nf); }

// Per-column statistics of one column held as values r_0 .. r_{n-1}:
// xbar = r_0 + (sum_{i>=1} (r_i - r_0)) / n   and   d = sum_i (r_i - xbar)^2  (fp32), and
// z = sum_{i>=1} |r_i - r_0|, which is zero exactly when all n values are equal.
template <int NMAX>
__device__ __forceinline__ void column_stats(const float* r, int n, float nf, float& xbar, float& d, float& z)
{
    const float base = r[0];
    float acc = 0.0f, spread = 0.0f;
#pragma unroll
    for (int i = 1; i < NMAX; ++i)
        if (i < n) {
            const float diff = r[i] - base;
            acc = acc + diff;
            spread = spread + fabsf(diff);
        }
    z = spread;
    xbar = base + mean_offset(acc, nf);
    float s = 0.0f;
#pragma unroll
    for (int i = 0; i < NMAX; ++i)
        if (i < n) {
            const float dev = r[i] - xbar;
            s = s + dev * dev;
        }
    d = s;
}

// A column's fp32 sum of squared deviations (or its loss term h t^2) is within about n 2^-24 of
// its exact value while it lies in [2^-100, 2^100]: no square in it has overflowed, and a square
// that underflowed (below 2^-126) is negligible beside the sum.  Outside that range -- deviations
// below about 2^-50 or above 2^50, an infinity, a NaN -- the column is recomputed in fp64 from the
// fp32 values, which holds for any fp32 input, unless the fp32 result is an exact zero.  The
// workloads stay in the range; the fp64 path (slow on this part) only runs for such columns.
__device__ __forceinline__ bool sum_sq_in_range(float s) { return s >= 0x1p-100f && s <= 0x1p100f; }

// A loss term l = (h t) t that is exactly zero because t = 0, or h = 0 with t finite.
__device__ __forceinline__ bool loss_term_exact_zero(float l, float h, float t)
{
    return l == 0.0f && (t == 0.0f || (h == 0.0f && fabsf(t) <= 0x1.fffffep127f));
}

// A loss term whose fp32 value can be used: in range (|l|, so that a negative curvature h takes
// no fp64 path either) or an exact zero.
__device__ __forceinline__ bool loss_term_usable(float l, float h, float t)
{
    return sum_sq_in_range(fabsf(l)) || loss_term_exact_zero(l, h, t);
}

// Whether every value get(i), i < n, equals xbar: with an fp32 sum of zero this makes the
// column's squared deviations exactly zero.
template <int NMAX, class Get>
__device__ __forceinline__ bool all_equal(const Get& get, int n, float xbar)
{
    const int m = NMAX > 0 ? NMAX : n;  // NMAX = 0: any n
    bool eq = true;
#pragma unroll
    for (int i = 0; i < m; ++i)
        if (i < n) eq = eq && get(i) == xbar;
    return eq;
}

// sum_i (get(i) - xbar)^2 in fp64.
template <int NMAX, class Get>
__device__ __forceinline__ double sq_dev_f64(const Get& get, int n, float xbar)
{
    const int m = NMAX > 0 ? NMAX : n;
    const double xb = (double)xbar;
    double s = 0.0;
#pragma unroll
    for (int i = 0; i < m; ++i)
        if (i < n) {
            const double dev = (double)get(i) - xb;
            s = s + dev * dev;
        }
    return s;
}

// A column's squared deviations from its fp32 sum d: d itself when usable, else fp64.
template <int NMAX, class Get>
__device__ __forceinline__ double checked_sq_dev(const Get& get, int n, float xbar, float d)
{
    if (sum_sq_in_range(d)) return (double)d;
    if (d == 0.0f && all_equal<NMAX>(get, n, xbar)) return 0.0;
    return sq_dev_f64<NMAX>(get, n, xbar);
}

// A column's loss term h (xbar - c)^2 (before the factor 1/2): the fp32 value when usable, else fp64.
__device__ __forceinline__ double checked_loss_term(float h, float xbar, float c)
{
    const float t = xbar - c;
    const float l = (h * t) * t;
    if (loss_term_usable(l, h, t)) return (double)l;
    const double td = (double)xbar - (double)c;
    return ((double)h * td) * td;
}

}  // namespace adpsgd
