// sync_step.cu -- the local step of a sync iteration fused with the averaging that ends it
// (Algorithm 2: the last "updating parameter variables locally" of an interval, then the
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

// Register cap: 128 per thread (2 blocks of 256 per SM) up to 8 replicas, 255 for 16.  One
// thread per column group.  Other forms measured slower on resnet18-n8 (0.316 ms here):
// - splitting a group's replicas over two lanes that swap halves by shuffles (0.346 ms);
// - a tiled form, with a thread per (group, replica) as in local_step_kernel and the averaging
//   from a shared-memory tile (0.350 ms);
// - the step over the replicas in chunks of 4 under a runtime loop, stashing the new x in shared
//   memory, to shrink the unrolled code (0.336 ms);
// - this form capped at 80 registers for 3 blocks per SM, which spills (0.426 ms);
// - 128-thread blocks at 96 registers, 5 per SM, no spills (0.337 ms).
template <int NMAX, bool BF16, bool LOSS>
__global__ void __launch_bounds__(kThreads, (NMAX >= 16 ? 1 : 2)) sync_step_kernel(const SyncStepParams p)
{
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
#pragma unroll
        for (int i = 0; i < NMAX; ++i)
            if (i < a.n) {
                const float4 z = BF16 ? make_float4(bf16_bits_to_float(nb[i].x & 0xFFFFu),
                                                    __uint_as_float(nb[i].x & 0xFFFF0000u),
                                                    bf16_bits_to_float(nb[i].y & 0xFFFFu),
                                                    __uint_as_float(nb[i].y & 0xFFFF0000u))
                                      : normals4(p.keys, (uint32_t)q + p.q0, (uint32_t)i, p.k, 0u);
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

// ------------------------------------------------------------------------------------------
// Pipelined form (Philox noise, 3..16 replicas): the loads go through shared memory by
// per-thread asynchronous copies (cp.async), so data in flight holds no registers.
// ------------------------------------------------------------------------------------------
// Each thread owns one float4 column group of all n replicas per iteration of a persistent
// grid-stride loop, as in sync_step_kernel.  Its shared-memory slots hold x_i and v_i of every
// replica i (and h, c), slot-major with the block's threads consecutive (conflict-free 16-byte
// accesses).  One commit group per replica: the copies of (group q, replica i) are waited for
// just before replica i is stepped, and as soon as it has been read its slots are refilled with
// (next group, replica i).  So while a thread steps the rest of group q and averages it, the
// copies for the next group are in flight: up to n * 32 bytes per thread without holding a
// register, on more resident warps than the register-resident form (whose loads held 2 n float4).
// The arithmetic is the local step's and the averaging's, in the same order (bit-identical).
constexpr int kPipeThreads = 128;

__device__ __forceinline__ void cp_async16(float4* smem_dst, const float4* gmem_src)
{
    const unsigned dst = (unsigned)__cvta_generic_to_shared(smem_dst);
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16;\n" ::"r"(dst), "l"(gmem_src) : "memory");
}

__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;\n" ::: "memory"); }

// Wait until at most N of this thread's most recent commit groups are still in flight.
template <int N>
__device__ __forceinline__ void cp_async_wait() { asm volatile("cp.async.wait_group %0;\n" ::"n"(N) : "memory"); }

template <int NMAX>
constexpr int pipe_slots() { return 2 * NMAX + 2; }  // x_i, v_i per replica, then h and c

// Issue the copies of (group q, replica i) into the thread's slots; h and c ride with replica 0.
// Out-of-range groups and inactive replicas issue nothing (their commit group stays empty).
template <int NMAX>
__device__ __forceinline__ void pipe_fill(const SyncStepParams& p, float4* slots, int64_t q, int i)
{
    const AvgParams& a = p.avg;
    if (q >= a.Q || i >= a.n) return;
    const int64_t row = (int64_t)i * a.P;
    cp_async16(slots + (2 * i) * kPipeThreads, reinterpret_cast<const float4*>(a.x + row) + q);
    cp_async16(slots + (2 * i + 1) * kPipeThreads, reinterpret_cast<const float4*>(p.v + row) + q);
    if (i == 0) {
        cp_async16(slots + (2 * NMAX) * kPipeThreads, reinterpret_cast<const float4*>(a.h) + q);
        cp_async16(slots + (2 * NMAX + 1) * kPipeThreads, reinterpret_cast<const float4*>(a.c) + q);
    }
}

template <int NMAX, bool LOSS>
__global__ void __launch_bounds__(kPipeThreads, (NMAX >= 16 ? 3 : 6)) sync_step_pipe_kernel(const SyncStepParams p)
{
    extern __shared__ float4 pipe_smem[];
    float4* slots = pipe_smem + threadIdx.x;  // slot s of this thread: slots[s * kPipeThreads]
    const AvgParams& a = p.avg;
    const float nf = (float)a.n;
    const bool wd = p.wd != 0.0f;
    double accD = 0.0, accL = 0.0;
    bool redo = false;
    const int64_t stride = (int64_t)gridDim.x * kPipeThreads;
    const int64_t q_first = (int64_t)blockIdx.x * kPipeThreads + threadIdx.x;
#pragma unroll
    for (int i = 0; i < NMAX; ++i) {
        pipe_fill<NMAX>(p, slots, q_first, i);
        cp_async_commit();
    }
    for (int64_t q = q_first; q < a.Q; q += stride) {
        const int64_t q_next = q + stride;
        float4 xv[NMAX];
        float4 hv = make_float4(0.0f, 0.0f, 0.0f, 0.0f), cv = hv;
#pragma unroll
        for (int i = 0; i < NMAX; ++i) {
            // Commit groups in flight: (q, i .. NMAX-1) then (q_next, 0 .. i-1); the oldest is (q, i).
            cp_async_wait<NMAX - 1>();
            if (i < a.n) {
                if (i == 0) {
                    hv = slots[(2 * NMAX) * kPipeThreads];
                    cv = slots[(2 * NMAX + 1) * kPipeThreads];
                }
                float4 x = slots[(2 * i) * kPipeThreads];
                float4 v = slots[(2 * i + 1) * kPipeThreads];
                const float4 z = normals4(p.keys, (uint32_t)q + p.q0, (uint32_t)i, p.k, 0u);
                if (wd) {
                    sgd_update<true>(x.x, v.x, hv.x, cv.x, z.x, p.gamma, p.mu, p.wd, p.sigma);
                    sgd_update<true>(x.y, v.y, hv.y, cv.y, z.y, p.gamma, p.mu, p.wd, p.sigma);
                    sgd_update<true>(x.z, v.z, hv.z, cv.z, z.z, p.gamma, p.mu, p.wd, p.sigma);
                    sgd_update<true>(x.w, v.w, hv.w, cv.w, z.w, p.gamma, p.mu, p.wd, p.sigma);
                } else {
                    sgd_update<false>(x.x, v.x, hv.x, cv.x, z.x, p.gamma, p.mu, p.wd, p.sigma);
                    sgd_update<false>(x.y, v.y, hv.y, cv.y, z.y, p.gamma, p.mu, p.wd, p.sigma);
                    sgd_update<false>(x.z, v.z, hv.z, cv.z, z.z, p.gamma, p.mu, p.wd, p.sigma);
                    sgd_update<false>(x.w, v.w, hv.w, cv.w, z.w, p.gamma, p.mu, p.wd, p.sigma);
                }
                reinterpret_cast<float4*>(p.v + (int64_t)i * a.P)[q] = v;
                xv[i] = x;
            } else {
                xv[i] = make_float4(0.0f, 0.0f, 0.0f, 0.0f);
            }
            // The slots of replica i have been read (the update used them): refill them.
            pipe_fill<NMAX>(p, slots, q_next, i);
            cp_async_commit();
        }
        redo |= !finish_group<NMAX, true, LOSS, true, true>(a, q, xv, nf, accD, accL);
    }
    cp_async_wait<0>();
    if (redo)
        for (int64_t q = q_first; q < a.Q; q += stride) redo_group<true, LOSS, true>(a, q, nf, accD, accL);
    finish_sums_n<LOSS, kPipeThreads>(a, accD, accL);
}

using SyncStepKernel = void (*)(const SyncStepParams);

template <int NMAX>
SyncStepKernel pick_nmax(bool bf16, bool loss)
{
    if (bf16) return loss ? sync_step_kernel<NMAX, true, true> : sync_step_kernel<NMAX, true, false>;
    return loss ? sync_step_kernel<NMAX, false, true> : sync_step_kernel<NMAX, false, false>;
}

// The launch form of a shape: the kernel, its block size and its dynamic shared memory.
struct SyncStepForm {
    SyncStepKernel kernel;
    int threads;
    size_t smem;
};

template <int NMAX>
SyncStepForm pipe_form(bool loss)
{
    const size_t smem = (size_t)pipe_slots<NMAX>() * kPipeThreads * sizeof(float4);
    return {loss ? sync_step_pipe_kernel<NMAX, true> : sync_step_pipe_kernel<NMAX, false>, kPipeThreads, smem};
}

// Philox noise with 3 to 16 replicas: the pipelined form.  Otherwise (up to 2 replicas, or the
// bf16 noise tensor) the register-resident form.
SyncStepForm pick(int32_t n, bool bf16, bool loss)
{
    if (!bf16 && n >= 3) {
        if (n <= 4) return pipe_form<4>(loss);
        if (n <= 8) return pipe_form<8>(loss);
        return pipe_form<16>(loss);
    }
    SyncStepKernel k;
    if (n <= 2) k = pick_nmax<2>(bf16, loss);
    else if (n <= 4) k = pick_nmax<4>(bf16, loss);
    else if (n <= 8) k = pick_nmax<8>(bf16, loss);
    else k = pick_nmax<16>(bf16, loss);
    return {k, kThreads, 0};
}

// Dynamic shared memory above the default 48 KB must be allowed per kernel before its launch.
cudaError_t allow_smem(const SyncStepForm& f)
{
    if (f.smem <= 48 * 1024) return cudaSuccess;
    return cudaFuncSetAttribute(f.kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)f.smem);
}

}  // namespace

// Used where it measured faster than the two kernels it replaces: up to 8 replicas, and up to 16
// with the pre-materialised bf16 noise.  With Philox noise and 9..16 replicas the 16-replica form
// (one block per SM, 8 warps) measured 0.04 to 0.41 ms slower per sync from P = 2^22 to 2^26.
bool sync_step_supported(int32_t n, int64_t P, const void* x, const void* v, const void* h, const void* c,
                         const void* noise_bf16)
{
    auto al = [](const void* ptr, unsigned mask) { return (reinterpret_cast<uintptr_t>(ptr) & mask) == 0; };
    const int max_n = noise_bf16 != nullptr ? kSyncStepMaxReplicas : 8;
    return n >= 1 && n <= max_n && P % 4 == 0 && al(x, 15) && al(v, 15) && al(h, 15) && al(c, 15) &&
           (noise_bf16 == nullptr || al(noise_bf16, 7));
}

int sync_step_grid(int32_t n, int64_t P, bool bf16, bool loss, int sms)
{
    const SyncStepForm f = pick(n, bf16, loss);
    int per_sm = 0;
    if (allow_smem(f) != cudaSuccess ||
        cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, f.kernel, f.threads, f.smem) != cudaSuccess ||
        per_sm < 1) {
        cudaGetLastError();
        per_sm = 1;
    }
    const int64_t work = (P / 4 + f.threads - 1) / f.threads;
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
    const SyncStepForm f = pick(s.n, s.noise_bf16 != nullptr, s.loss);
    const cudaError_t e = allow_smem(f);
    if (e != cudaSuccess) return e;
    f.kernel<<<(unsigned)s.grid, f.threads, f.smem, stream>>>(p);
    return cudaGetLastError();
}

}  // namespace adpsgd
