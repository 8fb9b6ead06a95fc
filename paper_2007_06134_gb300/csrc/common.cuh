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

// Fixed-order block sum over a block of kThreads threads; the result is valid in thread 0.
__device__ __forceinline__ double block_sum(double v, double* shared)
{
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) v += __shfl_down_sync(0xFFFFFFFFu, v, off);
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    if (lane == 0) shared[warp] = v;
    __syncthreads();
    double total = 0.0;
    if (threadIdx.x == 0)
        for (int w = 0; w < kThreads / 32; ++w) total += shared[w];
    __syncthreads();
    return total;
}

// Per-column statistics of one column held as values r_0 .. r_{n-1}:
// xbar = r_0 + (sum_{i>=1} (r_i - r_0)) / n   and   d = sum_i (r_i - xbar)^2  (fp32).
template <int NMAX>
__device__ __forceinline__ void column_stats(const float* r, int n, float nf, float& xbar, float& d)
{
    const float base = r[0];
    float acc = 0.0f;
#pragma unroll
    for (int i = 1; i < NMAX; ++i)
        if (i < n) acc = acc + (r[i] - base);
    xbar = base + __fdiv_rn(acc, nf);
    float s = 0.0f;
#pragma unroll
    for (int i = 0; i < NMAX; ++i)
        if (i < n) {
            const float dev = r[i] - xbar;
            s = s + dev * dev;
        }
    d = s;
}

}  // namespace adpsgd
