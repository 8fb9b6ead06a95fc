// kernels.cu -- sm_103a kernels of the ADPSGD hot path.
//
//   local_step_kernel  Algorithm 2's local update for all n replicas in
//                      one pass: gradient of the quadratic surrogate, Philox/Box-Muller noise
//                      (or a pre-materialised bf16 noise tensor), weight decay, momentum and
//                      the parameter update, 128-bit loads and stores.  HBM-bound: per
//                      replica-param it moves x and v in and out (16 B) plus h and c once
//                      per column (8/n B, re-reads across replicas hit L2).
//   average_kernel     Algorithm 2 averaging + S_k: per column, the replica mean, the squared
//                      deviations and the surrogate loss, x̄ written back to every replica;
//                      replica values of a column stay in registers between the passes.
//                      Persistent grid; each block leaves one fp64 partial per sum and the
//                      last block to finish adds them in block order (deterministic; an
//                      atomic ticket, no inter-block wait).  HBM-bound: 8 B per replica-param.
//   *_fill kernels     the raw Philox stream, its fp32 normals, and the bf16 noise tensor.
//
// The averaging's per-group arithmetic (mean, squared deviations, loss, the fp32-range guard and
// its second pass, the block sums) is in average.cuh, shared with sync_step_kernel
// (sync_step.cu), which fuses a sync iteration's local step with its averaging.
//
// Every fp32 operation of the update, the mean and the generator is written out once and
// compiled with -fmad=false, so results are bit-identical to any IEEE evaluation of the same
// sequence.
#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include <mutex>

#include "average.cuh"
#include "common.cuh"
#include "launch.h"
#include "noise.cuh"

namespace adpsgd {

void make_philox_keys(uint64_t seed, PhiloxKeys* out)
{
    uint32_t lo = (uint32_t)(seed & 0xFFFFFFFFull);
    uint32_t hi = (uint32_t)(seed >> 32);
    for (int r = 0; r < 10; ++r) {
        out->lo[r] = lo;
        out->hi[r] = hi;
        lo += 0x9E3779B9u;  // Weyl constants of Philox4x32
        hi += 0xBB67AE85u;
    }
}

namespace {

// ------------------------------------------------------------------------------------------
// Local step
// ------------------------------------------------------------------------------------------
struct StepParams {
    float* x;
    float* v;
    const float* h;
    const float* c;
    const uint16_t* noise;
    int64_t P;
    int64_t Q;  // ceil(P / 4): blocks of four elements, one Philox call each
    int32_t n;
    uint32_t k;
    uint32_t q0;  // Philox block of the first column: the column offset of a shard, divided by 4
    uint32_t r0;  // global index of replica 0 (the first replica of a replica split)
    float gamma, mu, wd, sigma;
    PhiloxKeys keys;
};

// Block b handles replica i = b mod n and the column groups (four columns each)
// q = (b div n) * kStepGroupsPerBlock + g * kStepThreads + tid, g < kStepGroups, so the n blocks
// that read the same h, c tile run back to back (the re-reads hit L2).  Each thread issues the
// loads of its kStepGroups groups before any arithmetic; 128-thread blocks with two groups per
// thread measured 5 % faster than 256 threads with one.
constexpr int kStepThreads = 128;
constexpr int kStepGroups = 2;
constexpr int kStepGroupsPerBlock = kStepThreads * kStepGroups;

template <bool VEC, bool BF16, bool WD>
__global__ void __launch_bounds__(kStepThreads) local_step_kernel(const StepParams p)
{
    const int64_t b = blockIdx.x;
    const int32_t i = (int32_t)(b % p.n);
    const int64_t q0 = (b / p.n) * kStepGroupsPerBlock + threadIdx.x;
    const int64_t row = (int64_t)i * p.P;
    if (VEC) {
        float4 xv[kStepGroups], vv[kStepGroups], hv[kStepGroups], cv[kStepGroups], zb[kStepGroups];
#pragma unroll
        for (int g = 0; g < kStepGroups; ++g) {
            const int64_t q = q0 + g * kStepThreads;
            if (q < p.Q) {
                xv[g] = reinterpret_cast<const float4*>(p.x + row)[q];
                vv[g] = reinterpret_cast<const float4*>(p.v + row)[q];
                hv[g] = __ldg(reinterpret_cast<const float4*>(p.h) + q);
                cv[g] = __ldg(reinterpret_cast<const float4*>(p.c) + q);
                if (BF16) {
                    const uint2 nb = __ldg(reinterpret_cast<const uint2*>(p.noise + row) + q);
                    zb[g] = make_float4(bf16_bits_to_float(nb.x & 0xFFFFu), __uint_as_float(nb.x & 0xFFFF0000u),
                                        bf16_bits_to_float(nb.y & 0xFFFFu), __uint_as_float(nb.y & 0xFFFF0000u));
                }
            }
        }
#pragma unroll
        for (int g = 0; g < kStepGroups; ++g) {
            const int64_t q = q0 + g * kStepThreads;
            if (q >= p.Q) break;
            const float4 z = BF16 ? zb[g] : normals4(p.keys, (uint32_t)q + p.q0, (uint32_t)i + p.r0, p.k, 0u);
            sgd_update<WD>(xv[g].x, vv[g].x, hv[g].x, cv[g].x, z.x, p.gamma, p.mu, p.wd, p.sigma);
            sgd_update<WD>(xv[g].y, vv[g].y, hv[g].y, cv[g].y, z.y, p.gamma, p.mu, p.wd, p.sigma);
            sgd_update<WD>(xv[g].z, vv[g].z, hv[g].z, cv[g].z, z.z, p.gamma, p.mu, p.wd, p.sigma);
            sgd_update<WD>(xv[g].w, vv[g].w, hv[g].w, cv[g].w, z.w, p.gamma, p.mu, p.wd, p.sigma);
            reinterpret_cast<float4*>(p.x + row)[q] = xv[g];
            reinterpret_cast<float4*>(p.v + row)[q] = vv[g];
        }
    } else {
        for (int g = 0; g < kStepGroups; ++g) {
            const int64_t q = q0 + g * kStepThreads;
            if (q >= p.Q) break;
            float zz[4];
            if (!BF16) {
                const float4 z = normals4(p.keys, (uint32_t)q + p.q0, (uint32_t)i + p.r0, p.k, 0u);
                zz[0] = z.x; zz[1] = z.y; zz[2] = z.z; zz[3] = z.w;
            }
#pragma unroll
            for (int r = 0; r < 4; ++r) {
                const int64_t j = 4 * q + r;
                if (j >= p.P) break;
                float xs = p.x[row + j];
                float vs = p.v[row + j];
                const float z = BF16 ? bf16_bits_to_float(p.noise[row + j]) : zz[r];
                sgd_update<WD>(xs, vs, __ldg(p.h + j), __ldg(p.c + j), z, p.gamma, p.mu, p.wd, p.sigma);
                p.x[row + j] = xs;
                p.v[row + j] = vs;
            }
        }
    }
}

// ------------------------------------------------------------------------------------------
// Averaging + variance (the per-group arithmetic is in average.cuh)
// ------------------------------------------------------------------------------------------
// Persistent grid over column groups; each thread keeps the n replica values of U groups in
// registers (NMAX >= n), so the loads of U groups are in flight together.  NMAX = 0: any n,
// values re-read per pass, fp64 inline where a column needs it.  The block partials are added
// by the last block to finish, in block order, so the sums do not depend on which block
// finishes last.
template <int NMAX, int U, bool VEC, bool LOSS, bool WRITE>
__global__ void __launch_bounds__(kThreads, ((NMAX == 2 || (NMAX <= 8 && U == 1)) ? 4 : (NMAX >= 32 ? 1 : 2)))
    average_kernel(const AvgParams p)
{
    using G = ColumnGroup<VEC>;
    using T = typename G::T;
    const float nf = (float)p.n;
    double accD = 0.0, accL = 0.0;
    bool redo = false;  // finish_group refused a group of this thread
    const int64_t stride = (int64_t)gridDim.x * kThreads;
    for (int64_t q0 = (int64_t)blockIdx.x * kThreads + threadIdx.x; q0 < p.Q; q0 += U * stride) {
        if (NMAX > 0) {
            constexpr int R = NMAX > 0 ? NMAX : 1;
            T vals[U][R];
#pragma unroll
            for (int u = 0; u < U; ++u) {
                const int64_t q = q0 + u * stride;
                if (q < p.Q) {
#pragma unroll
                    for (int i = 0; i < R; ++i)
                        if (i < p.n) vals[u][i] = reinterpret_cast<const T*>(p.x + (int64_t)i * p.P)[q];
                }
            }
#pragma unroll
            for (int u = 0; u < U; ++u) {
                const int64_t q = q0 + u * stride;
                if (q < p.Q) redo |= !finish_group<R, VEC, LOSS, WRITE>(p, q, vals[u], nf, accD, accL);
            }
        } else {
            const int64_t q = q0;
            float xbar[G::W];
#pragma unroll
            for (int r = 0; r < G::W; ++r) {
                const int64_t j = G::W * q + r;
                float d, z;
                column_stats_global(p.x, p.P, j, p.n, nf, xbar[r], d, z);
                accD += checked_sq_dev<0>([&](int i) { return p.x[(int64_t)i * p.P + j]; }, p.n, xbar[r], d);
                if (LOSS) accL += checked_loss_term(p.h[j], xbar[r], p.c[j]);
            }
            if (WRITE) {
                const T out = G::make(xbar);
                for (int i = 0; i < p.n; ++i) reinterpret_cast<T*>(p.x + (int64_t)i * p.P)[q] = out;
            }
        }
    }
    if (NMAX > 0 && redo)
        for (int64_t q = (int64_t)blockIdx.x * kThreads + threadIdx.x; q < p.Q; q += stride)
            redo_group<VEC, LOSS, WRITE>(p, q, nf, accD, accL);
    finish_sums<LOSS>(p, accD, accL);
}

// ------------------------------------------------------------------------------------------
// Generator fills
// ------------------------------------------------------------------------------------------
__global__ void __launch_bounds__(kThreads) philox_fill_kernel(PhiloxKeys keys, uint32_t tag, int32_t n,
                                                               int64_t nq, uint32_t k, uint4* out)
{
    const int64_t t = (int64_t)blockIdx.x * kThreads + threadIdx.x;
    if (t >= (int64_t)n * nq) return;
    const uint32_t i = (uint32_t)(t / nq);
    const uint32_t q = (uint32_t)(t % nq);
    out[t] = philox4x32_10(make_uint4(q, i, k, tag), keys);
}

__global__ void __launch_bounds__(kThreads) noise_f32_kernel(PhiloxKeys keys, uint32_t tag, int32_t n,
                                                             int64_t P, int64_t Q, uint32_t k, float* out)
{
    const int64_t t = (int64_t)blockIdx.x * kThreads + threadIdx.x;
    if (t >= (int64_t)n * Q) return;
    const int64_t i = t / Q, q = t % Q;
    const float4 z = normals4(keys, (uint32_t)q, (uint32_t)i, k, tag);
    const float zz[4] = {z.x, z.y, z.z, z.w};
#pragma unroll
    for (int r = 0; r < 4; ++r)
        if (4 * q + r < P) out[i * P + 4 * q + r] = zz[r];
}

__global__ void __launch_bounds__(kThreads) noise_bf16_kernel(PhiloxKeys keys, int32_t n, int64_t P,
                                                              int64_t Q, uint32_t r0, uint32_t q0, uint16_t* out)
{
    const int64_t t = (int64_t)blockIdx.x * kThreads + threadIdx.x;
    if (t >= (int64_t)n * Q) return;
    const int64_t i = t / Q, q = t % Q;
    const float4 z = normals4(keys, (uint32_t)q + q0, (uint32_t)i + r0, 0u, 1u);
    const float zz[4] = {z.x, z.y, z.z, z.w};
#pragma unroll
    for (int r = 0; r < 4; ++r)
        if (4 * q + r < P) out[i * P + 4 * q + r] = __bfloat16_as_ushort(__float2bfloat16_rn(zz[r]));
}

template <typename Kernel>
int max_blocks_per_sm(Kernel kernel)
{
    int nb = 0;
    if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&nb, kernel, kThreads, 0) != cudaSuccess) {
        cudaGetLastError();
        nb = 1;
    }
    return nb < 1 ? 1 : nb;
}

using AvgKernel = void (*)(const AvgParams);

template <int NMAX, int U, int UL = U>
AvgKernel pick_average_nmax(bool vec, bool loss, bool write)
{
    // UL: groups per thread of the variant with the loss (h and c take registers too)
    if (vec) {
        if (!write) return average_kernel<NMAX, U, true, false, false>;
        return loss ? average_kernel<NMAX, UL, true, true, true> : average_kernel<NMAX, U, true, false, true>;
    }
    if (!write) return average_kernel<NMAX, U, false, false, false>;
    return loss ? average_kernel<NMAX, UL, false, true, true> : average_kernel<NMAX, U, false, false, true>;
}

// Register-resident variants: NMAX replicas x U column groups per thread (NMAX * U <= 32 float4).
// Resident blocks per SM (the register cap): 4 for n <= 2 and for one group per thread up to 8
// replicas, 1 for n <= 32 and 2 otherwise.  With
// two rows per column a thread has few bytes in flight, so n <= 2 takes 4 blocks of 4 groups:
// measured 0.93 of the copy peak at P = 2^28, against 0.71 with 2 blocks.  Its loss variant takes
// 2 groups, which fit the 64 registers of that cap without spilling.  For 3 to 8 replicas, 4
// blocks of one group per thread measured (L2 flushed; P = 2^22 / 2^24 / 2^26 / 2^28)
// 0.79 / 0.92 / 0.96 / 0.96 of the copy peak at n = 4 and 0.89 / 0.92 / 0.93 / 0.94 at n = 8, against
// 0.65 / 0.87 / 0.95 / 0.98 and 0.85 / 0.91 / 0.92 / 0.92 with 2 blocks of 4 and of 2 groups.  With
// the loss (h and c read too) the one-group form measured slower right after a local step (0.92
// against 0.96 of the peak on 8 replicas of 138 M columns), so the loss variants keep 2 blocks of
// 4 (n <= 4) and 2 (n <= 8) groups.  For 16 replicas 3 blocks measured 0.89-0.90 against 0.92 with 2.
AvgKernel pick_average(int32_t n, bool vec, bool loss, bool write)
{
    if (n <= 2) return pick_average_nmax<2, 4, 2>(vec, loss, write);
    if (n <= 4) return pick_average_nmax<4, 1, 4>(vec, loss, write);
    if (n <= 8) return pick_average_nmax<8, 1, 2>(vec, loss, write);
    if (n <= 16) return pick_average_nmax<16, 1>(vec, loss, write);
    if (n <= 32) return pick_average_nmax<32, 1>(vec, loss, write);
    return pick_average_nmax<0, 1>(vec, loss, write);
}

bool use_vec(int64_t P, const void* a, const void* b, const void* c, const void* d)
{
    auto al = [](const void* ptr) { return ptr == nullptr || (reinterpret_cast<uintptr_t>(ptr) & 15u) == 0; };
    return (P % 4 == 0) && al(a) && al(b) && al(c) && al(d);
}

int64_t ceil_div(int64_t a, int64_t b) { return (a + b - 1) / b; }

}  // namespace

cudaError_t launch_local_step(const LocalStepArgs& a, cudaStream_t stream)
{
    StepParams p;
    p.x = a.x;
    p.v = a.v;
    p.h = a.h;
    p.c = a.c;
    p.noise = a.noise_bf16;
    p.P = a.P;
    p.Q = ceil_div(a.P, 4);
    p.n = a.n;
    p.k = a.k;
    p.q0 = a.q0;
    p.r0 = a.r0;
    p.gamma = a.gamma;
    p.mu = a.mu;
    p.wd = a.wd;
    p.sigma = a.sigma;
    p.keys = *a.keys;
    const bool vec = use_vec(a.P, a.x, a.v, a.h, a.c) &&
                     (a.noise_bf16 == nullptr || (reinterpret_cast<uintptr_t>(a.noise_bf16) & 7u) == 0);
    const bool bf16 = a.noise_bf16 != nullptr;
    const bool wd = a.wd != 0.0f;
    const int64_t blocks = (int64_t)a.n * ceil_div(p.Q, kStepGroupsPerBlock);
    void (*kernel)(const StepParams);
    if (vec) {
        if (bf16) kernel = wd ? local_step_kernel<true, true, true> : local_step_kernel<true, true, false>;
        else kernel = wd ? local_step_kernel<true, false, true> : local_step_kernel<true, false, false>;
    } else {
        if (bf16) kernel = wd ? local_step_kernel<false, true, true> : local_step_kernel<false, true, false>;
        else kernel = wd ? local_step_kernel<false, false, true> : local_step_kernel<false, false, false>;
    }
    kernel<<<(unsigned)blocks, kStepThreads, 0, stream>>>(p);
    return cudaGetLastError();
}

int average_grid_max(int sms) { return sms * (2048 / kThreads); }

int average_grid(int32_t n, int64_t P, bool loss, bool write_back, int sms)
{
    // vector-ness does not change the occupancy enough to matter; size for the vector kernel
    const AvgKernel kernel = pick_average(n, true, loss, write_back);
    const int per_sm = max_blocks_per_sm(kernel);
    const int64_t work = ceil_div(ceil_div(P, 4), kThreads);
    int64_t grid = (int64_t)per_sm * sms;
    if (grid > work) grid = work;
    if (grid < 1) grid = 1;
    const int cap = average_grid_max(sms);
    return (int)(grid > cap ? cap : grid);
}

cudaError_t launch_average(const AverageArgs& a, cudaStream_t stream)
{
    const bool loss = a.h != nullptr;
    const bool vec = use_vec(a.P, a.x, a.h, a.c, nullptr);
    AvgParams p;
    p.x = a.x;
    p.h = a.h;
    p.c = a.c;
    p.P = a.P;
    p.Q = vec ? a.P / 4 : a.P;
    p.n = a.n;
    p.partials = a.partials;
    p.out = a.out;
    p.counter = a.counter;
    const AvgKernel kernel = pick_average(a.n, vec, loss, a.write_back);
    kernel<<<a.grid, kThreads, 0, stream>>>(p);
    return cudaGetLastError();
}

cudaError_t launch_philox_fill(uint64_t seed, uint32_t tag, int32_t n, int64_t nq, uint32_t k,
                               uint32_t* out, cudaStream_t stream)
{
    PhiloxKeys keys;
    make_philox_keys(seed, &keys);
    const int64_t blocks = ceil_div((int64_t)n * nq, kThreads);
    if (blocks == 0) return cudaSuccess;
    philox_fill_kernel<<<(unsigned)blocks, kThreads, 0, stream>>>(keys, tag, n, nq, k, reinterpret_cast<uint4*>(out));
    return cudaGetLastError();
}

cudaError_t launch_noise_f32(uint64_t seed, uint32_t tag, int32_t n, int64_t P, uint32_t k, float* out,
                             cudaStream_t stream)
{
    PhiloxKeys keys;
    make_philox_keys(seed, &keys);
    const int64_t Q = ceil_div(P, 4);
    const int64_t blocks = ceil_div((int64_t)n * Q, kThreads);
    if (blocks == 0) return cudaSuccess;
    noise_f32_kernel<<<(unsigned)blocks, kThreads, 0, stream>>>(keys, tag, n, P, Q, k, out);
    return cudaGetLastError();
}

cudaError_t launch_noise_bf16(uint64_t seed, int32_t n, int64_t P, uint32_t r0, uint32_t q0, uint16_t* out,
                              cudaStream_t stream)
{
    PhiloxKeys keys;
    make_philox_keys(seed, &keys);
    const int64_t Q = ceil_div(P, 4);
    const int64_t blocks = ceil_div((int64_t)n * Q, kThreads);
    if (blocks == 0) return cudaSuccess;
    noise_bf16_kernel<<<(unsigned)blocks, kThreads, 0, stream>>>(keys, n, P, Q, r0, q0, out);
    return cudaGetLastError();
}

// ------------------------------------------------------------------------------------------
// Fixed device scratch for the averaging entry point that allocates nothing
// ------------------------------------------------------------------------------------------
// The partial sums of up to kStaticMaxBlocks blocks (D then loss), the two finished sums and one
// slot for the completion counter: 2 * 2048 + 4 doubles = 32.8 KB, held by every GPU that loads
// this library until exit.
constexpr int kStaticMaxBlocks = 2048;
constexpr int kStaticMaxDevices = 64;

}  // namespace adpsgd

static __device__ __align__(256) double g_static_scratch[2 * adpsgd::kStaticMaxBlocks + 4];

namespace adpsgd {

namespace {

std::mutex g_static_mutex;

// The address of g_static_scratch as seen by one CUDA context.  A module's globals move when its
// context is destroyed and created again (cudaDeviceReset, a primary-context reset, or another
// context made current), so the cached address is tied to the context's process-unique id.
struct StaticAddress {
    unsigned long long context_id = 0;
    double* address = nullptr;
};
StaticAddress g_static_address[kStaticMaxDevices];

using CtxGetIdFn = CUresult (*)(CUcontext, unsigned long long*);

// Id of the current context (cuCtxGetId with a null context), found through the runtime's
// driver entry-point lookup so that the library needs no link against the driver library.
cudaError_t current_context_id(unsigned long long* id)
{
    static CtxGetIdFn get_id = nullptr;
    static bool looked_up = false;
    if (!looked_up) {
        void* fn = nullptr;
        cudaDriverEntryPointQueryResult found = cudaDriverEntryPointSymbolNotFound;
        const cudaError_t e = cudaGetDriverEntryPointByVersion("cuCtxGetId", &fn, 12000, cudaEnableDefault, &found);
        if (e != cudaSuccess) return e;
        if (found != cudaDriverEntryPointSuccess || fn == nullptr) return cudaErrorSymbolNotFound;
        get_id = reinterpret_cast<CtxGetIdFn>(fn);
        looked_up = true;
    }
    return get_id(nullptr, id) == CUDA_SUCCESS ? cudaSuccess : cudaErrorDeviceUninitialized;
}

}  // namespace

int static_scratch_max_blocks() { return kStaticMaxBlocks; }

// Device address of g_static_scratch in the current device's current context.  In host code the
// symbol's name is only a stand-in, not a device address, so the address is looked up with
// cudaGetSymbolAddress (with that device current) the first time a context calls, and cached
// with the context's id.  cudaGetSymbolAddress also creates the runtime's context if there is
// none yet, so the id is read after it on a first call.
cudaError_t static_scratch_address(double** partials, double** out, unsigned int** counter)
{
    int device = 0;
    cudaError_t e = cudaGetDevice(&device);
    if (e != cudaSuccess) return e;
    if (device < 0 || device >= kStaticMaxDevices) return cudaErrorInvalidDevice;
    std::lock_guard<std::mutex> lock(g_static_mutex);
    StaticAddress& slot = g_static_address[device];
    unsigned long long id = 0;
    const bool have_id = current_context_id(&id) == cudaSuccess;
    if (!have_id || slot.address == nullptr || slot.context_id != id) {
        void* address = nullptr;
        e = cudaGetSymbolAddress(&address, g_static_scratch);
        if (e != cudaSuccess) return e;
        e = current_context_id(&id);
        if (e != cudaSuccess) return e;
        slot.context_id = id;
        slot.address = static_cast<double*>(address);
    }
    *partials = slot.address;
    *out = slot.address + 2 * kStaticMaxBlocks;
    *counter = reinterpret_cast<unsigned int*>(slot.address + 2 * kStaticMaxBlocks + 2);
    return cudaSuccess;
}

}  // namespace adpsgd
