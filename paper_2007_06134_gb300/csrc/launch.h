// launch.h -- internal interface between the host runtime and the CUDA kernels.
#pragma once

#include <cuda_runtime_api.h>

#include <cstdint>

namespace adpsgd {

// Round keys of Philox4x32-10 for one seed: key r = key 0 + r * (Weyl constants).
struct PhiloxKeys {
    uint32_t lo[10];
    uint32_t hi[10];
};

// Round keys of Philox4x32-10 for a 64-bit seed (key = (seed lo, seed hi), bumped by the
// Weyl constants once per round).
void make_philox_keys(uint64_t seed, PhiloxKeys* out);

// One local step of every replica (Algorithm 2, update line).
struct LocalStepArgs {
    float* x;
    float* v;
    const float* h;
    const float* c;
    const uint16_t* noise_bf16;  // nullptr: Philox noise
    const PhiloxKeys* keys;
    int32_t n;
    int64_t P;
    uint32_t k;
    uint32_t q0;  // Philox block of column 0 (a shard's column offset / 4; 0 unsharded)
    uint32_t r0;  // global index of replica 0 (a replica split's first replica; 0 otherwise)
    float gamma, mu, wd, sigma;
};
cudaError_t launch_local_step(const LocalStepArgs& a, cudaStream_t stream);

// Averaging + variance (+ loss): per-block fp64 partials, added in block order by the last
// block to finish into out[0] (D) and out[1] (loss).  *counter must be zero at launch; the
// kernel leaves it zero.
struct AverageArgs {
    float* x;
    const float* h;  // nullptr unless the loss is wanted
    const float* c;
    int32_t n;
    int64_t P;
    bool write_back;  // false: variance only
    double* partials; // 2 * grid doubles
    double* out;      // 2 doubles
    unsigned int* counter;
    int grid;         // from average_grid()
};
cudaError_t launch_average(const AverageArgs& a, cudaStream_t stream);
// Blocks of the persistent averaging kernel for this shape on a device with `sms` SMs.
int average_grid(int32_t n, int64_t P, bool loss, bool write_back, int sms);
int average_grid_max(int sms);

// The local step of a sync iteration fused with the averaging that ends it: the same results
// as launch_local_step followed by launch_average (write-back, loss when h_loss is set), with
// out[0] = D and out[1] = loss as there.  Needs sync_step_supported().
constexpr int kSyncStepMaxReplicas = 16;
struct SyncStepArgs {
    float* x;
    float* v;
    const float* h;
    const float* c;
    const uint16_t* noise_bf16;  // nullptr: Philox noise
    const PhiloxKeys* keys;
    int32_t n;
    int64_t P;
    uint32_t k;
    uint32_t q0;       // Philox block of column 0
    float gamma, mu, wd, sigma;
    bool loss;
    double* partials;  // 2 * grid doubles
    double* out;       // 2 doubles
    unsigned int* counter;
    int grid;          // from sync_step_grid()
};
bool sync_step_supported(int32_t n, int64_t P, const void* x, const void* v, const void* h, const void* c,
                         const void* noise_bf16);
int sync_step_grid(int32_t n, int64_t P, bool bf16, bool loss, int sms);
cudaError_t launch_sync_step(const SyncStepArgs& a, cudaStream_t stream);

// bytes from src to dst by a copy kernel on `stream`.  Both are device addresses (for host
// memory: the mapped device address of a page-locked buffer), 16-byte aligned.
cudaError_t launch_copy(void* dst, const void* src, int64_t bytes, int sms, cudaStream_t stream);
// dst rows [0, rows) of P floats each (row stride P) = the P floats at src, a device address (for
// host memory: the mapped device address of a page-locked buffer); src may be one of dst's rows.
cudaError_t launch_broadcast_rows(float* dst, const float* src, int32_t rows, int64_t P, int sms, cudaStream_t stream);

// Fixed device scratch (no allocation): partial sums for up to static_scratch_max_blocks()
// blocks, the two finished sums and the completion counter.  The first call on a device looks the address up.
int static_scratch_max_blocks();
cudaError_t static_scratch_address(double** partials, double** out, unsigned int** counter);

// A fused sync interval: m (<= kMaxFusedSteps) local steps of every replica from step k0 with
// step sizes gamma[0..m), then (average) the averaging with its sums in out[0..1].  n <= 32.
constexpr int kMaxFusedSteps = 256;
struct IntervalArgs {
    float* x;
    float* v;
    const float* h;
    const float* c;
    const uint16_t* noise_bf16;
    const PhiloxKeys* keys;
    int32_t n;
    int64_t P;
    uint32_t k0;
    uint32_t q0;         // Philox block of column 0
    int32_t m;
    const float* gamma;  // host array of m step sizes
    float mu, wd, sigma;
    bool average;
    bool loss;
    double* partials;  // 2 * grid
    double* out;
    unsigned int* counter;
    int grid;  // from interval_grid()
};
cudaError_t launch_interval(const IntervalArgs& a, cudaStream_t stream);
int interval_grid(int32_t n, int64_t P, int sms);
int interval_grid_max(int sms);
int interval_max_replicas();

cudaError_t launch_philox_fill(uint64_t seed, uint32_t tag, int32_t n, int64_t nq, uint32_t k,
                               uint32_t* out, cudaStream_t stream);
cudaError_t launch_noise_f32(uint64_t seed, uint32_t tag, int32_t n, int64_t P, uint32_t k,
                             float* out, cudaStream_t stream);
// Rows [r0, r0 + n) and columns [4 q0, 4 q0 + P) of the bf16 noise tensor of the whole problem.
cudaError_t launch_noise_bf16(uint64_t seed, int32_t n, int64_t P, uint32_t r0, uint32_t q0, uint16_t* out,
                              cudaStream_t stream);

}  // namespace adpsgd
