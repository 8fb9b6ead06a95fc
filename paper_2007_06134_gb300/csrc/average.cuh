// average.cuh -- the averaging arithmetic shared by average_kernel (kernels.cu) and
// sync_step_kernel (sync_step.cu): per column group, the replica mean, the squared deviations and
// the loss in fp32 with the fp32-range guard, the write-back of the mean, the second pass over
// refused groups, and the deterministic block sums.
#pragma once

#include <cstdint>

#include "common.cuh"

namespace adpsgd {
namespace {

struct AvgParams {
    float* x;
    const float* h;
    const float* c;
    int64_t P;
    int64_t Q;  // column groups: blocks of four columns (vector) or single columns (scalar)
    int32_t n;
    double* partials;       // 2 * gridDim.x: per-block D, then per-block loss
    double* out;            // out[0] = D, out[1] = loss
    unsigned int* counter;  // zero at launch; the last block to finish sets it back to zero
};

// Columns with more than 32 replicas: the same arithmetic, re-reading x (L1/L2) per pass.
__device__ __forceinline__ void column_stats_global(const float* x, int64_t P, int64_t j, int n, float nf,
                                                    float& xbar, float& d, float& z)
{
    const float base = x[j];
    float acc = 0.0f, spread = 0.0f;
    for (int i = 1; i < n; ++i) {
        const float diff = x[(int64_t)i * P + j] - base;
        acc = acc + diff;
        spread = spread + fabsf(diff);
    }
    z = spread;
    xbar = base + mean_offset(acc, nf);
    float s = 0.0f;
    for (int i = 0; i < n; ++i) {
        const float dev = x[(int64_t)i * P + j] - xbar;
        s = s + dev * dev;
    }
    d = s;
}

// A column group is one float4 (four columns) of every replica, or one float (scalar rows).
template <bool VEC> struct ColumnGroup;
template <> struct ColumnGroup<true> {
    using T = float4;
    static constexpr int W = 4;
    static __device__ __forceinline__ float lane(const float4& v, int r)
    {
        return r == 0 ? v.x : (r == 1 ? v.y : (r == 2 ? v.z : v.w));
    }
    static __device__ __forceinline__ float4 make(const float* f) { return make_float4(f[0], f[1], f[2], f[3]); }
};
template <> struct ColumnGroup<false> {
    using T = float;
    static constexpr int W = 1;
    static __device__ __forceinline__ float lane(float v, int) { return v; }
    static __device__ __forceinline__ float make(const float* f) { return f[0]; }
};

// A column group's fp32 sums can be added as they are when each lies in the accurate range of
// sum_sq_in_range or is an exact zero: the squared deviations d when every column's values are all
// equal (z = 0), the loss terms when each is zero because t = 0, or h = 0 with t finite.  The
// first pass (finish_group) adds a group's d and writes it back when d is usable, and adds its
// loss when both are usable.  The second pass (redo_group) recomputes the same decisions and adds
// the rest.
template <int W>
__device__ __forceinline__ float group_sum(const float* a)
{
    return W == 4 ? (a[0] + a[W > 1 ? 1 : 0]) + (a[W > 2 ? 2 : 0] + a[W > 3 ? 3 : 0]) : a[0];
}

template <int W>
__device__ __forceinline__ bool dev_usable(const float* d, const float* z)
{
    const float dsum = group_sum<W>(d);
    return sum_sq_in_range(dsum) || (dsum == 0.0f && group_sum<W>(z) == 0.0f);
}

template <int W>
__device__ __forceinline__ bool loss_usable(const float* l, const float* hs, const float* ts)
{
    if (sum_sq_in_range(fabsf(group_sum<W>(l)))) return true;
    bool zero = true;
#pragma unroll
    for (int r = 0; r < W; ++r) zero = zero && loss_term_exact_zero(l[r], hs[r], ts[r]);
    return zero;
}

// Statistics, loss and write-back of column group q whose replica values are vals[0..n), all in
// fp32 and without branches.  Returns false when part of the group is left to redo_group.
// STORE_REFUSED: vals are not yet in x (they come from a local step in registers), so a group
// whose d is refused has vals written to x instead of the mean, for redo_group to start from.
template <int R, bool VEC, bool LOSS, bool WRITE, bool STORE_REFUSED = false>
__device__ __forceinline__ bool finish_group(const AvgParams& p, int64_t q, const typename ColumnGroup<VEC>::T* vals,
                                             float nf, double& accD, double& accL)
{
    using G = ColumnGroup<VEC>;
    constexpr int W = G::W;
    float xbar[W], d[W], z[W];
#pragma unroll
    for (int r = 0; r < W; ++r) {
        float col[R];
#pragma unroll
        for (int i = 0; i < R; ++i) col[i] = (i < p.n) ? G::lane(vals[i], r) : 0.0f;
        column_stats<R>(col, p.n, nf, xbar[r], d[r], z[r]);
    }
    const bool d_ok = dev_usable<W>(d, z);
    if (d_ok) accD += (double)group_sum<W>(d);
    bool l_ok = true;
    if (LOSS) {
        const typename G::T hv = reinterpret_cast<const typename G::T*>(p.h)[q];
        const typename G::T cv = reinterpret_cast<const typename G::T*>(p.c)[q];
        float l[W], hs[W], ts[W];
#pragma unroll
        for (int r = 0; r < W; ++r) {
            hs[r] = G::lane(hv, r);
            ts[r] = xbar[r] - G::lane(cv, r);
            l[r] = (hs[r] * ts[r]) * ts[r];
        }
        l_ok = loss_usable<W>(l, hs, ts);
        if (d_ok && l_ok) accL += (double)group_sum<W>(l);
    }
    if (WRITE && d_ok) {
        const typename G::T out = G::make(xbar);
#pragma unroll
        for (int i = 0; i < R; ++i)
            if (i < p.n) reinterpret_cast<typename G::T*>(p.x + (int64_t)i * p.P)[q] = out;
    }
    if (STORE_REFUSED && !d_ok) {
#pragma unroll
        for (int i = 0; i < R; ++i)
            if (i < p.n) reinterpret_cast<typename G::T*>(p.x + (int64_t)i * p.P)[q] = vals[i];
    }
    return d_ok && l_ok;
}

// Second pass over a thread's column groups, run only by threads for which finish_group returned
// false.  The same fp32 arithmetic on x decides again.  A group whose d was usable was added (and
// written back: its columns now all equal their mean, which averaging leaves unchanged, so d is
// usable again and the mean and loss terms are the same); only a loss finish_group left out is
// added here.  A group whose d was refused is still unchanged in x; it is redone here column by
// column, with fp64 where a column needs it, and written back.
template <bool VEC, bool LOSS, bool WRITE>
__device__ void redo_group(const AvgParams& p, int64_t q, float nf, double& accD, double& accL)
{
    using G = ColumnGroup<VEC>;
    constexpr int W = G::W;
    float xbar[W], d[W], z[W], l[W], hs[W], ts[W];
    for (int r = 0; r < W; ++r) {
        const int64_t j = W * q + r;
        column_stats_global(p.x, p.P, j, p.n, nf, xbar[r], d[r], z[r]);
        if (LOSS) {
            hs[r] = p.h[j];
            ts[r] = xbar[r] - p.c[j];
            l[r] = (hs[r] * ts[r]) * ts[r];
        }
    }
    const bool d_ok = dev_usable<W>(d, z);
    const bool l_ok = !LOSS || loss_usable<W>(l, hs, ts);
    if (d_ok && l_ok) return;
    for (int r = 0; r < W; ++r) {
        const int64_t j = W * q + r;
        if (!d_ok) accD += checked_sq_dev<0>([&](int i) { return p.x[(int64_t)i * p.P + j]; }, p.n, xbar[r], d[r]);
        if (LOSS) accL += checked_loss_term(p.h[j], xbar[r], p.c[j]);
    }
    if (WRITE && !d_ok)
        for (int r = 0; r < W; ++r)
            for (int i = 0; i < p.n; ++i) p.x[(int64_t)i * p.P + W * q + r] = xbar[r];
}

// The end of a persistent averaging kernel of THREADS-thread blocks: each block leaves its fp64
// partials of D and the loss; the last block to finish (an atomic ticket, no inter-block wait)
// adds them in block order into out[0] = D and out[1] = loss / 2, and resets the ticket.
// Deterministic for a given grid.
template <bool LOSS, int THREADS>
__device__ __forceinline__ void finish_sums_n(const AvgParams& p, double accD, double accL)
{
    __shared__ double shared[THREADS / 32];
    __shared__ unsigned int ticket;
    const double bD = block_sum<THREADS>(accD, shared);
    const double bL = LOSS ? block_sum<THREADS>(accL, shared) : 0.0;
    if (threadIdx.x == 0) {
        p.partials[blockIdx.x] = bD;
        p.partials[gridDim.x + blockIdx.x] = bL;
        __threadfence();
        ticket = atomicAdd(p.counter, 1u);
    }
    __syncthreads();
    if (ticket != gridDim.x - 1) return;
    // The last block: every other block's partials are visible (fence before each increment).
    __threadfence();
    double d = 0.0, l = 0.0;
    for (int b = threadIdx.x; b < (int)gridDim.x; b += THREADS) {
        d += __ldcg(p.partials + b);
        if (LOSS) l += __ldcg(p.partials + gridDim.x + b);
    }
    d = block_sum<THREADS>(d, shared);
    if (LOSS) l = block_sum<THREADS>(l, shared);
    if (threadIdx.x == 0) {
        p.out[0] = d;
        p.out[1] = 0.5 * l;
        *p.counter = 0u;
    }
}

template <bool LOSS>
__device__ __forceinline__ void finish_sums(const AvgParams& p, double accD, double accL)
{
    finish_sums_n<LOSS, kThreads>(p, accD, accL);
}

}  // namespace
}  // namespace adpsgd
