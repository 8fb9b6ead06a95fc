// sync_step.cu -- the local step of a sync iteration fused with the averaging that ends it
// (Algorithm 2: the last local update of an interval, then the
// averaging and S_k).  Each thread owns one float4 column group of all n replicas: it loads x,
// v (and h, c once), applies the local step to every replica in registers with the same
// operations as local_step_kernel, writes v, and then averages the new x with the same
// operations as average_kernel (average.cuh).  Per replica-param that moves 16 B (+8/n) instead
// of the 25 B of the two kernels run one after the other, since x is not written and read
// back in between.  Nothing here depends on the objective being separable across steps: only
// the update of one iteration is fused with the averaging that follows it.
#include <cuda_runtime.h>

#include <cstdint>

#include "average.cuh"
#include "common.cuh"
#include "launch.h"
#include "noise.cuh"

namespace adpsgd {
namespace {

struct SyncStepParams {
    AvgParams avg;          // x, h, c, P, Q = P / 4, n, partials, out, counter
    float* v;
    const uint16_t* noise;  // pre-materialised bf16 noise [n, P], or nullptr (Philox)
    uint32_t k;
    uint32_t q0;            // Philox block of column 0
    float gamma, mu, wd, sigma;
    PhiloxKeys keys;
};

// Register cap: 128 per thread (2 blocks of 256 per SM) up to 8 replicas, 255 for 16, and 85 (3
// blocks) for 3-4 replicas with Philox noise, which measured 0.90 against 0.87 of the copy peak at
// n = 3, P = 2^26 (0.94 against 0.93 at n = 4); 2 replicas fit 3 blocks at the 128 cap.  One
// thread per column group.  With Philox noise the n normals4 calls run first, in a loop that is
// not unrolled, into per-thread shared-memory slots (NMAX x 256 float4 per block): the
// generator's code is there once instead of n times, and its arithmetic runs while the loads of
// x and v are in flight.  Against the same kernel with the generator unrolled into the update
// (below the register-resident form of the list) it measured 0.93 against 0.84 of the copy peak
// at n = 8, P = 2^26, 0.90 against 0.81 at 2^24 and 0.93 against 0.87 at n = 4, P = 2^26.  The
// two-halves form below, with halves of 4 at 5 or 6 blocks of 128 per SM (92 or 80 registers),
// measured 0.85-0.86 at n = 8, P = 2^26 and 0.80 at n = 6, against 0.93 and 0.88 here; the
// generator loop unrolled by two (two replicas' chains interleaved) measured 0.5-1.5 % slower,
// and v staged in shared memory by per-thread cp.async copies while the generator runs (79-96
// registers: 2 or 3 blocks of 256, or 5 or 6 of 128 per SM) 0.80-0.90 against 0.92 at n = 8.
// Other forms measured slower on resnet18-n8 than the unrolled form did at the time (0.314 ms,
// one launch under ncu, 225 M warp-instructions at 60 % issue; 0.294 ms and 213 M since the
// generator's fma division and square root):
// - splitting a group's replicas over two lanes that swap halves by shuffles (0.346 ms);
// - a tiled form, with a thread per (group, replica) as in local_step_kernel and the averaging
//   from a shared-memory tile (0.350 ms);
// - the step over the replicas in chunks of 4 under a runtime loop, stashing the new x in shared
//   memory, to shrink the unrolled code (0.336 ms);
// - this form capped at 80 registers for 3 blocks per SM, which spills (0.426 ms);
// - 128-thread blocks at 96 registers, 5 per SM, no spills (0.337 ms);
// - loads streamed through shared memory by per-thread cp.async copies, refilled replica by
//   replica for the next group, 6 blocks of 128 per SM: 0.333 ms with the replicas unrolled
//   (250 M instructions, instruction-fetch stalls 2.0 per issue), 0.314 ms with a replica loop
//   that is not unrolled (258 M instructions at 72 % issue: the copies' per-thread address work
//   takes what the higher issue rate gains);
// - a tile per block with a barrier, each thread stepping two (replica, group) items and then
//   averaging whole columns of the tile: 0.469 ms (400 M instructions);
// - per-warp bulk copies (cp.async.bulk on mbarriers, lane 0 refilling a 3-stage ring): 0.396 ms
//   (351 M instructions, most of the excess in the waits);
// - v loaded one replica ahead instead of with x (78 registers, 3 blocks of 256 per SM): 0.75 of
//   the copy peak at n = 8, P = 2^26, against 0.79 here;
// - (after the generator's fma division and square root, which brought this form to 0.85 there)
//   the replicas in a loop that is not unrolled, the next replica's x and v loaded into registers
//   while one is stepped, the new x in per-thread shared-memory slots: 0.77-0.79 at 6 or 8 blocks
//   of 128 per SM;
// - teams of 8 lanes over two column groups, lane i stepping replica i as local_step_kernel does
//   (80 registers, 3 blocks of 256 per SM), the new x through a shared-memory tile and lane j
//   then taking column j's mean and squared deviations, with shuffles for the group sums: 0.360 ms
//   under ncu, 306 M instructions (per-lane statistics, shuffles and h, c loads), 0.56 of the copy
//   peak at n = 8, P = 2^26, and 0.45 with bf16 noise; 4 blocks per SM (64 registers) was slower.
template <int NMAX, bool BF16, bool LOSS>
__global__ void __launch_bounds__(kThreads, (NMAX >= 16 ? 1 : ((NMAX == 4 && !BF16) ? 3 : 2)))
    sync_step_kernel(const SyncStepParams p)
{
    __shared__ float4 zs[BF16 ? 1 : NMAX][BF16 ? 1 : kThreads];  // thread t's normals of replica i: zs[i][t]
    const AvgParams& a = p.avg;
    const float nf = (float)a.n;
    const bool wd = p.wd != 0.0f;
    double accD = 0.0, accL = 0.0;
    bool redo = false;
    const int64_t stride = (int64_t)gridDim.x * kThreads;
    for (int64_t q = (int64_t)blockIdx.x * kThreads + threadIdx.x; q < a.Q; q += stride) {
        float4 xv[NMAX], vv[NMAX];
        uint2 nb[NMAX];
        const float4 hv = __ldg(reinterpret_cast<const float4*>(a.h) + q);
        const float4 cv = __ldg(reinterpret_cast<const float4*>(a.c) + q);
#pragma unroll
        for (int i = 0; i < NMAX; ++i)
            if (i < a.n) {
                const int64_t row = (int64_t)i * a.P;
                xv[i] = reinterpret_cast<const float4*>(a.x + row)[q];
                vv[i] = reinterpret_cast<const float4*>(p.v + row)[q];
                if (BF16) nb[i] = __ldg(reinterpret_cast<const uint2*>(p.noise + row) + q);
            }
        if (!BF16) {
#pragma unroll 1
            for (int i = 0; i < a.n; ++i)
                zs[i][threadIdx.x] = normals4(p.keys, (uint32_t)q + p.q0, (uint32_t)i, p.k, 0u);
        }
#pragma unroll
        for (int i = 0; i < NMAX; ++i)
            if (i < a.n) {
                const float4 z = BF16 ? make_float4(bf16_bits_to_float(nb[i].x & 0xFFFFu),
                                                    __uint_as_float(nb[i].x & 0xFFFF0000u),
                                                    bf16_bits_to_float(nb[i].y & 0xFFFFu),
                                                    __uint_as_float(nb[i].y & 0xFFFF0000u))
                                      : zs[i][threadIdx.x];
                if (wd) {
                    sgd_update<true>(xv[i].x, vv[i].x, hv.x, cv.x, z.x, p.gamma, p.mu, p.wd, p.sigma);
                    sgd_update<true>(xv[i].y, vv[i].y, hv.y, cv.y, z.y, p.gamma, p.mu, p.wd, p.sigma);
                    sgd_update<true>(xv[i].z, vv[i].z, hv.z, cv.z, z.z, p.gamma, p.mu, p.wd, p.sigma);
                    sgd_update<true>(xv[i].w, vv[i].w, hv.w, cv.w, z.w, p.gamma, p.mu, p.wd, p.sigma);
                } else {
                    sgd_update<false>(xv[i].x, vv[i].x, hv.x, cv.x, z.x, p.gamma, p.mu, p.wd, p.sigma);
                    sgd_update<false>(xv[i].y, vv[i].y, hv.y, cv.y, z.y, p.gamma, p.mu, p.wd, p.sigma);
                    sgd_update<false>(xv[i].z, vv[i].z, hv.z, cv.z, z.z, p.gamma, p.mu, p.wd, p.sigma);
                    sgd_update<false>(xv[i].w, vv[i].w, hv.w, cv.w, z.w, p.gamma, p.mu, p.wd, p.sigma);
                }
                reinterpret_cast<float4*>(p.v + (int64_t)i * a.P)[q] = vv[i];
            }
        redo |= !finish_group<NMAX, true, LOSS, true, true>(a, q, xv, nf, accD, accL);
    }
    if (redo)
        for (int64_t q = (int64_t)blockIdx.x * kThreads + threadIdx.x; q < a.Q; q += stride)
            redo_group<true, LOSS, true>(a, q, nf, accD, accL);
    finish_sums<LOSS>(a, accD, accL);
}

using SyncStepKernel = void (*)(const SyncStepParams);

// 9..16 replicas with Philox noise: the replicas in two halves of up to 8.  For each half the
// thread loads x and v into registers, draws the half's normals in a rolled loop into its
// shared-memory slots, applies the update, writes v and puts the new x into the same slots.
// The averaging then takes the n new values of the group from shared memory.  Registers hold
// one half at a time, so 4 blocks of 128 threads (16 warps) fit per SM where the 16-replica
// register form fits 8 warps.  Same operations and order as sync_step_kernel.  Balanced halves
// (n = 9 as 5 + 4, 12 as 6 + 6) measured 1-3 % slower than 8 first.  With the bf16 noise tensor
// this form (spilling a few registers) measured 0.87-0.95 against 0.90-0.96 for the 16-replica
// register form, which has no generator to hide.
constexpr int kHalvesThreads = 128;
constexpr int kHalf = 8;

template <bool LOSS>
__global__ void __launch_bounds__(kHalvesThreads, 4) sync_step_halves_kernel(const SyncStepParams p)
{
    // thread t, replica i: slots[t][i]; the pad row keeps the 16-byte accesses of 8 neighbouring
    // threads on distinct banks
    __shared__ float4 slots[kHalvesThreads][2 * kHalf + 1];
    const AvgParams& a = p.avg;
    const float nf = (float)a.n;
    const bool wd = p.wd != 0.0f;
    const int t = threadIdx.x;
    double accD = 0.0, accL = 0.0;
    bool redo = false;
    const int64_t stride = (int64_t)gridDim.x * kHalvesThreads;
    for (int64_t q = (int64_t)blockIdx.x * kHalvesThreads + t; q < a.Q; q += stride) {
        const float4 hv = __ldg(reinterpret_cast<const float4*>(a.h) + q);
        const float4 cv = __ldg(reinterpret_cast<const float4*>(a.c) + q);
#pragma unroll 1
        for (int r0 = 0; r0 < a.n; r0 += kHalf) {
            float4 xv[kHalf], vv[kHalf];
#pragma unroll
            for (int u = 0; u < kHalf; ++u)
                if (r0 + u < a.n) {
                    const int64_t row = (int64_t)(r0 + u) * a.P;
                    xv[u] = reinterpret_cast<const float4*>(a.x + row)[q];
                    vv[u] = reinterpret_cast<const float4*>(p.v + row)[q];
                }
#pragma unroll 1
            for (int i = r0; i < a.n && i < r0 + kHalf; ++i)
                slots[t][i] = normals4(p.keys, (uint32_t)q + p.q0, (uint32_t)i, p.k, 0u);
#pragma unroll
            for (int u = 0; u < kHalf; ++u)
                if (r0 + u < a.n) {
                    const float4 z = slots[t][r0 + u];
                    if (wd) {
                        sgd_update<true>(xv[u].x, vv[u].x, hv.x, cv.x, z.x, p.gamma, p.mu, p.wd, p.sigma);
                        sgd_update<true>(xv[u].y, vv[u].y, hv.y, cv.y, z.y, p.gamma, p.mu, p.wd, p.sigma);
                        sgd_update<true>(xv[u].z, vv[u].z, hv.z, cv.z, z.z, p.gamma, p.mu, p.wd, p.sigma);
                        sgd_update<true>(xv[u].w, vv[u].w, hv.w, cv.w, z.w, p.gamma, p.mu, p.wd, p.sigma);
                    } else {
                        sgd_update<false>(xv[u].x, vv[u].x, hv.x, cv.x, z.x, p.gamma, p.mu, p.wd, p.sigma);
                        sgd_update<false>(xv[u].y, vv[u].y, hv.y, cv.y, z.y, p.gamma, p.mu, p.wd, p.sigma);
                        sgd_update<false>(xv[u].z, vv[u].z, hv.z, cv.z, z.z, p.gamma, p.mu, p.wd, p.sigma);
                        sgd_update<false>(xv[u].w, vv[u].w, hv.w, cv.w, z.w, p.gamma, p.mu, p.wd, p.sigma);
                    }
                    reinterpret_cast<float4*>(p.v + (int64_t)(r0 + u) * a.P)[q] = vv[u];
                    slots[t][r0 + u] = xv[u];
                }
        }
        redo |= !finish_group<2 * kHalf, true, LOSS, true, true>(a, q, slots[t], nf, accD, accL);
    }
    if (redo)
        for (int64_t q = (int64_t)blockIdx.x * kHalvesThreads + t; q < a.Q; q += stride)
            redo_group<true, LOSS, true>(a, q, nf, accD, accL);
    finish_sums_n<LOSS, kHalvesThreads>(a, accD, accL);
}

bool use_halves(int32_t n, bool bf16) { return !bf16 && n > kHalf && n <= 2 * kHalf; }

template <int NMAX>
SyncStepKernel pick_nmax(bool bf16, bool loss)
{
    if (bf16) return loss ? sync_step_kernel<NMAX, true, true> : sync_step_kernel<NMAX, true, false>;
    return loss ? sync_step_kernel<NMAX, false, true> : sync_step_kernel<NMAX, false, false>;
}

// 9..16 replicas: the two-halves form with Philox noise, the 16-replica register form with the
// bf16 noise tensor.
SyncStepKernel pick(int32_t n, bool bf16, bool loss)
{
    if (use_halves(n, bf16)) return loss ? sync_step_halves_kernel<true> : sync_step_halves_kernel<false>;
    if (n <= 2) return pick_nmax<2>(bf16, loss);
    if (n <= 4) return pick_nmax<4>(bf16, loss);
    if (n <= 8) return pick_nmax<8>(bf16, loss);
    return loss ? sync_step_kernel<16, true, true> : sync_step_kernel<16, true, false>;
}

}  // namespace

// Every shape it takes measured faster than the two kernels it replaces.  With Philox noise and
// 9..16 replicas the two-halves form measured 0.69-0.76 of the copy peak at n = 9, 0.77-0.83 at
// n = 12 and 0.83-0.89 at n = 16 (P = 2^22 to 2^26), against 0.56-0.64 for the two kernels; the
// 16-replica register form (one block of 256 per SM, 234 registers) had measured 0.54-0.66 there.
bool sync_step_supported(int32_t n, int64_t P, const void* x, const void* v, const void* h, const void* c,
                         const void* noise_bf16)
{
    auto al = [](const void* ptr, unsigned mask) { return (reinterpret_cast<uintptr_t>(ptr) & mask) == 0; };
    return n >= 1 && n <= kSyncStepMaxReplicas && P % 4 == 0 && al(x, 15) && al(v, 15) && al(h, 15) && al(c, 15) &&
           (noise_bf16 == nullptr || al(noise_bf16, 7));
}

int sync_step_grid(int32_t n, int64_t P, bool bf16, bool loss, int sms)
{
    const int threads = use_halves(n, bf16) ? kHalvesThreads : kThreads;
    int per_sm = 0;
    if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, pick(n, bf16, loss), threads, 0) != cudaSuccess ||
        per_sm < 1) {
        cudaGetLastError();
        per_sm = 1;
    }
    const int64_t work = (P / 4 + threads - 1) / threads;
    int64_t grid = (int64_t)per_sm * sms;
    if (grid > work) grid = work;
    if (grid < 1) grid = 1;
    const int cap = average_grid_max(sms);
    return (int)(grid > cap ? cap : grid);
}

cudaError_t launch_sync_step(const SyncStepArgs& s, cudaStream_t stream)
{
    SyncStepParams p;
    p.avg.x = s.x;
    p.avg.h = s.h;
    p.avg.c = s.c;
    p.avg.P = s.P;
    p.avg.Q = s.P / 4;
    p.avg.n = s.n;
    p.avg.partials = s.partials;
    p.avg.out = s.out;
    p.avg.counter = s.counter;
    p.v = s.v;
    p.noise = s.noise_bf16;
    p.k = s.k;
    p.q0 = s.q0;
    p.gamma = s.gamma;
    p.mu = s.mu;
    p.wd = s.wd;
    p.sigma = s.sigma;
    p.keys = *s.keys;
    const SyncStepKernel kernel = pick(s.n, s.noise_bf16 != nullptr, s.loss);
    kernel<<<(unsigned)s.grid, use_halves(s.n, s.noise_bf16 != nullptr) ? kHalvesThreads : kThreads, 0, stream>>>(p);
    return cudaGetLastError();
}

}  // namespace adpsgd
