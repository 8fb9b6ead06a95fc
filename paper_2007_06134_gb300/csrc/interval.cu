// interval.cu -- temporal fusion of one sync interval: m local steps of every replica followed
// by the averaging, in one kernel (Algorithm 2's inner loop between two syncs).
//
// The surrogate objective is separable per column, so each thread can keep the x and v of its
// four columns of one replica in registers for all m steps; only the averaging couples the
// replicas of a column, through shared memory, where every thread of the block takes a share of
// the tile's 128 columns.  Per replica-param the interval moves 16 bytes
// (x, v in and out) plus 8/n for h and c instead of 16 m + 8: the kernel is bound by the noise
// generator's arithmetic, not by HBM.  Every element goes through exactly the operations of
// local_step_kernel and average_kernel in the same order, so results are bit-identical to the
// unfused path.  A real model's gradient couples its parameters, so this only applies to
// separable objectives.
#include <cuda_runtime.h>

#include "common.cuh"
#include "launch.h"
#include "noise.cuh"

namespace adpsgd {

namespace {

constexpr int kTileGroups = 32;  // blockDim.x: groups of four columns per tile
constexpr int kMaxReplicas = 32; // blockDim.y = n <= 32

struct IntervalParams {
    float* x;
    float* v;
    const float* h;
    const float* c;
    const uint16_t* noise;
    int64_t P;
    int64_t Q;  // ceil(P / 4)
    int32_t n;
    uint32_t k0;
    uint32_t q0;  // Philox block of column 0
    int32_t m;
    float mu, wd, sigma;
    double* partials;
    double* out;
    unsigned int* counter;
    PhiloxKeys keys;
    float gamma[kMaxFusedSteps];
};

// Fixed-order sum over a block of any size (a multiple of 32 threads); valid in thread 0.
__device__ __forceinline__ double block_sum_any(double v, double* shared)
{
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) v += __shfl_down_sync(0xFFFFFFFFu, v, off);
    const int tid = threadIdx.y * blockDim.x + threadIdx.x;
    const int warps = (blockDim.x * blockDim.y) >> 5;
    if ((tid & 31) == 0) shared[tid >> 5] = v;
    __syncthreads();
    double total = 0.0;
    if (tid == 0)
        for (int w = 0; w < warps; ++w) total += shared[w];
    __syncthreads();
    return total;
}

// column_stats (common.cuh) for lane r of column group g, reading the n replica values from the
// shared tile: the same operations in the same order.
__device__ __forceinline__ void column_stats_tile(const float4 (*tile)[kTileGroups], int g, int r, int n, float nf,
                                                  float& xbar, float& d)
{
    const float base = reinterpret_cast<const float*>(&tile[0][g])[r];
    float acc = 0.0f;
    for (int j = 1; j < n; ++j) acc = acc + (reinterpret_cast<const float*>(&tile[j][g])[r] - base);
    xbar = base + mean_offset(acc, nf);
    float s = 0.0f;
    for (int j = 0; j < n; ++j) {
        const float dev = reinterpret_cast<const float*>(&tile[j][g])[r] - xbar;
        s = s + dev * dev;
    }
    d = s;
}

// Block (32, n): thread (g, i) owns columns 4q .. 4q+3 of replica i, q = tile * 32 + g.
template <bool VEC, bool BF16, bool WD, bool AVG, bool LOSS>
__global__ void __launch_bounds__(kTileGroups * kMaxReplicas) interval_kernel(const IntervalParams p)
{
    __shared__ float4 tile[kMaxReplicas][kTileGroups];
    __shared__ float4 xbar_s[kTileGroups];
    __shared__ float4 h_s[kTileGroups];
    __shared__ float4 c_s[kTileGroups];
    __shared__ double shared[kMaxReplicas];
    __shared__ unsigned int ticket;
    const int g = threadIdx.x;
    const int i = threadIdx.y;
    const int tid = threadIdx.y * blockDim.x + threadIdx.x;
    const int nthreads = blockDim.x * blockDim.y;
    const int n = p.n;
    const float nf = (float)n;
    double accD = 0.0, accL = 0.0;
    for (int64_t base = (int64_t)blockIdx.x * kTileGroups; base < p.Q; base += (int64_t)gridDim.x * kTileGroups) {
        const int64_t q = base + g;
        const bool active = q < p.Q;
        const int64_t row = (int64_t)i * p.P;
        const int valid = active ? (int)((p.P - 4 * q) < 4 ? (p.P - 4 * q) : 4) : 0;
        float xs[4] = {0.f, 0.f, 0.f, 0.f}, vs[4] = {0.f, 0.f, 0.f, 0.f};
        float hs[4] = {0.f, 0.f, 0.f, 0.f}, cs[4] = {0.f, 0.f, 0.f, 0.f};
        float zb[4] = {0.f, 0.f, 0.f, 0.f};
        if (VEC && active) {
            const float4 x4 = reinterpret_cast<const float4*>(p.x + row)[q];
            const float4 v4 = reinterpret_cast<const float4*>(p.v + row)[q];
            const float4 h4 = __ldg(reinterpret_cast<const float4*>(p.h) + q);
            const float4 c4 = __ldg(reinterpret_cast<const float4*>(p.c) + q);
            xs[0] = x4.x; xs[1] = x4.y; xs[2] = x4.z; xs[3] = x4.w;
            vs[0] = v4.x; vs[1] = v4.y; vs[2] = v4.z; vs[3] = v4.w;
            hs[0] = h4.x; hs[1] = h4.y; hs[2] = h4.z; hs[3] = h4.w;
            cs[0] = c4.x; cs[1] = c4.y; cs[2] = c4.z; cs[3] = c4.w;
            if (BF16) {
                const uint2 nb = __ldg(reinterpret_cast<const uint2*>(p.noise + row) + q);
                zb[0] = bf16_bits_to_float(nb.x & 0xFFFFu);
                zb[1] = __uint_as_float(nb.x & 0xFFFF0000u);
                zb[2] = bf16_bits_to_float(nb.y & 0xFFFFu);
                zb[3] = __uint_as_float(nb.y & 0xFFFF0000u);
            }
        } else if (!VEC) {
#pragma unroll
            for (int r = 0; r < 4; ++r)
                if (r < valid) {
                    const int64_t j = 4 * q + r;
                    xs[r] = p.x[row + j];
                    vs[r] = p.v[row + j];
                    hs[r] = __ldg(p.h + j);
                    cs[r] = __ldg(p.c + j);
                    if (BF16) zb[r] = bf16_bits_to_float(p.noise[row + j]);
                }
        }
        if (active) {
            for (int s = 0; s < p.m; ++s) {
                float z[4];
                if (BF16) {
                    z[0] = zb[0]; z[1] = zb[1]; z[2] = zb[2]; z[3] = zb[3];
                } else {
                    const float4 z4 = normals4(p.keys, (uint32_t)q + p.q0, (uint32_t)i, p.k0 + (uint32_t)s, 0u);
                    z[0] = z4.x; z[1] = z4.y; z[2] = z4.z; z[3] = z4.w;
                }
                const float gamma = p.gamma[s];
#pragma unroll
                for (int r = 0; r < 4; ++r) sgd_update<WD>(xs[r], vs[r], hs[r], cs[r], z[r], gamma, p.mu, p.wd, p.sigma);
            }
            if (VEC) {
                reinterpret_cast<float4*>(p.v + row)[q] = make_float4(vs[0], vs[1], vs[2], vs[3]);
                if (!AVG) reinterpret_cast<float4*>(p.x + row)[q] = make_float4(xs[0], xs[1], xs[2], xs[3]);
            } else {
#pragma unroll
                for (int r = 0; r < 4; ++r)
                    if (r < valid) {
                        p.v[row + 4 * q + r] = vs[r];
                        if (!AVG) p.x[row + 4 * q + r] = xs[r];
                    }
            }
        }
        if (!AVG) continue;
        tile[i][g] = make_float4(xs[0], xs[1], xs[2], xs[3]);
        if (LOSS && i == 0) {
            h_s[g] = make_float4(hs[0], hs[1], hs[2], hs[3]);
            c_s[g] = make_float4(cs[0], cs[1], cs[2], cs[3]);
        }
        __syncthreads();
        // The 128 columns of the tile are shared out over the whole block: thread t takes
        // columns t, t + 32n, ...; column col is lane col % 4 of group col / 4, so consecutive
        // threads read consecutive words of the tile.
        for (int col = tid; col < 4 * kTileGroups; col += nthreads) {
            const int cg = col >> 2, r = col & 3;
            const int64_t j = 4 * (base + cg) + r;
            if (base + cg >= p.Q || j >= p.P) continue;
            float xb, d;
            column_stats_tile(tile, cg, r, n, nf, xb, d);
            accD += checked_sq_dev<0>([&](int t) { return reinterpret_cast<const float*>(&tile[t][cg])[r]; }, n, xb, d);
            if (LOSS)
                accL += checked_loss_term(reinterpret_cast<const float*>(&h_s[cg])[r], xb,
                                          reinterpret_cast<const float*>(&c_s[cg])[r]);
            reinterpret_cast<float*>(xbar_s)[col] = xb;
        }
        __syncthreads();
        if (active) {
            const float4 xb = xbar_s[g];
            if (VEC) {
                reinterpret_cast<float4*>(p.x + row)[q] = xb;
            } else {
                const float xv[4] = {xb.x, xb.y, xb.z, xb.w};
#pragma unroll
                for (int r = 0; r < 4; ++r)
                    if (r < valid) p.x[row + 4 * q + r] = xv[r];
            }
        }
        __syncthreads();
    }
    if (!AVG) return;
    const double bD = block_sum_any(accD, shared);
    const double bL = LOSS ? block_sum_any(accL, shared) : 0.0;
    if (tid == 0) {
        p.partials[blockIdx.x] = bD;
        p.partials[gridDim.x + blockIdx.x] = bL;
        __threadfence();
        ticket = atomicAdd(p.counter, 1u);
    }
    __syncthreads();
    if (ticket != gridDim.x - 1) return;
    __threadfence();
    double d = 0.0, l = 0.0;
    for (int b = tid; b < (int)gridDim.x; b += nthreads) {
        d += __ldcg(p.partials + b);
        if (LOSS) l += __ldcg(p.partials + gridDim.x + b);
    }
    d = block_sum_any(d, shared);
    if (LOSS) l = block_sum_any(l, shared);
    if (tid == 0) {
        p.out[0] = d;
        p.out[1] = 0.5 * l;
        *p.counter = 0u;
    }
}

using IntervalKernel = void (*)(const IntervalParams);

template <bool VEC, bool BF16, bool WD>
IntervalKernel pick_interval3(bool avg, bool loss)
{
    if (!avg) return interval_kernel<VEC, BF16, WD, false, false>;
    return loss ? interval_kernel<VEC, BF16, WD, true, true> : interval_kernel<VEC, BF16, WD, true, false>;
}

IntervalKernel pick_interval(bool vec, bool bf16, bool wd, bool avg, bool loss)
{
    if (vec) {
        if (bf16) return wd ? pick_interval3<true, true, true>(avg, loss) : pick_interval3<true, true, false>(avg, loss);
        return wd ? pick_interval3<true, false, true>(avg, loss) : pick_interval3<true, false, false>(avg, loss);
    }
    if (bf16) return wd ? pick_interval3<false, true, true>(avg, loss) : pick_interval3<false, true, false>(avg, loss);
    return wd ? pick_interval3<false, false, true>(avg, loss) : pick_interval3<false, false, false>(avg, loss);
}

}  // namespace

int interval_max_replicas() { return kMaxReplicas; }

int interval_grid(int32_t n, int64_t P, int sms)
{
    const IntervalKernel kernel = pick_interval(true, false, true, true, true);
    int per_sm = 0;
    if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, kernel, kTileGroups * n, 0) != cudaSuccess) {
        cudaGetLastError();
        per_sm = 1;
    }
    if (per_sm < 1) per_sm = 1;
    const int64_t tiles = ((P + 3) / 4 + kTileGroups - 1) / kTileGroups;
    int64_t grid = (int64_t)per_sm * sms;
    if (grid > tiles) grid = tiles;
    if (grid < 1) grid = 1;
    const int cap = interval_grid_max(sms);
    return (int)(grid > cap ? cap : grid);
}

int interval_grid_max(int sms) { return sms * 32; }

cudaError_t launch_interval(const IntervalArgs& a, cudaStream_t stream)
{
    if (a.m < 1 || a.m > kMaxFusedSteps || a.n < 1 || a.n > kMaxReplicas) return cudaErrorInvalidValue;
    IntervalParams p;
    p.x = a.x;
    p.v = a.v;
    p.h = a.h;
    p.c = a.c;
    p.noise = a.noise_bf16;
    p.P = a.P;
    p.Q = (a.P + 3) / 4;
    p.n = a.n;
    p.k0 = a.k0;
    p.q0 = a.q0;
    p.m = a.m;
    p.mu = a.mu;
    p.wd = a.wd;
    p.sigma = a.sigma;
    p.partials = a.partials;
    p.out = a.out;
    p.counter = a.counter;
    p.keys = *a.keys;
    for (int s = 0; s < kMaxFusedSteps; ++s) p.gamma[s] = s < a.m ? a.gamma[s] : 0.0f;
    auto al = [](const void* ptr) { return ptr == nullptr || (reinterpret_cast<uintptr_t>(ptr) & 15u) == 0; };
    const bool vec = (a.P % 4 == 0) && al(a.x) && al(a.v) && al(a.h) && al(a.c) &&
                     (a.noise_bf16 == nullptr || (reinterpret_cast<uintptr_t>(a.noise_bf16) & 7u) == 0);
    const IntervalKernel kernel = pick_interval(vec, a.noise_bf16 != nullptr, a.wd != 0.0f, a.average, a.loss);
    kernel<<<a.grid, dim3(kTileGroups, a.n), 0, stream>>>(p);
    return cudaGetLastError();
}

}  // namespace adpsgd
