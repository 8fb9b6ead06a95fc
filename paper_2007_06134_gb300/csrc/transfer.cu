// transfer.cu -- host <-> device copies carried out by the SMs: a grid-stride copy kernel that
// reads or writes page-locked host memory through its mapped device address, and a broadcast of
// one row to every replica row (the initial model of every replica).  The copy engines
// queue few requests at a time, so their throughput drops with the host memory's latency when
// other work loads it; thousands of threads keep enough requests in flight to hide it.
#include <cuda_runtime.h>

#include <cstdint>

#include "launch.h"

namespace adpsgd {
namespace {

constexpr int kCopyThreads = 512;

// dst[i] = src[i] for i < n16 (16-byte words), four independent loads in flight per thread,
// then the last `tail` (< 16) bytes by thread 0 of block 0.
__global__ void __launch_bounds__(kCopyThreads) copy16_kernel(uint4* __restrict__ dst, const uint4* __restrict__ src,
                                                              int64_t n16, int tail)
{
    const int64_t stride = (int64_t)gridDim.x * kCopyThreads;
    int64_t i = (int64_t)blockIdx.x * kCopyThreads + threadIdx.x;
    for (; i + 3 * stride < n16; i += 4 * stride) {
        const uint4 a = src[i];
        const uint4 b = src[i + stride];
        const uint4 c = src[i + 2 * stride];
        const uint4 d = src[i + 3 * stride];
        dst[i] = a;
        dst[i + stride] = b;
        dst[i + 2 * stride] = c;
        dst[i + 3 * stride] = d;
    }
    for (; i < n16; i += stride) dst[i] = src[i];
    if (tail > 0 && blockIdx.x == 0 && threadIdx.x == 0) {
        unsigned char* db = reinterpret_cast<unsigned char*>(dst + n16);
        const unsigned char* sb = reinterpret_cast<const unsigned char*>(src + n16);
        for (int t = 0; t < tail; ++t) db[t] = sb[t];
    }
}

// dst row r (r < rows, row stride ld words) = src, for words [0, count): src is read once, four
// independent loads in flight per thread, each word written to every row.  src may be device
// memory or the mapped device address of page-locked host memory, and may be one of dst's rows
// (each word is read before any row of it is written, by the same thread).
template <typename T>
__global__ void __launch_bounds__(kCopyThreads) broadcast_rows_kernel(T* dst, const T* src, int32_t rows, int64_t ld,
                                                                      int64_t count)
{
    const int64_t stride = (int64_t)gridDim.x * kCopyThreads;
    int64_t i = (int64_t)blockIdx.x * kCopyThreads + threadIdx.x;
    for (; i + 3 * stride < count; i += 4 * stride) {
        const T a = src[i];
        const T b = src[i + stride];
        const T c = src[i + 2 * stride];
        const T d = src[i + 3 * stride];
        for (int32_t r = 0; r < rows; ++r) {
            T* row = dst + (int64_t)r * ld;
            row[i] = a;
            row[i + stride] = b;
            row[i + 2 * stride] = c;
            row[i + 3 * stride] = d;
        }
    }
    for (; i < count; i += stride) {
        const T a = src[i];
        for (int32_t r = 0; r < rows; ++r) dst[(int64_t)r * ld + i] = a;
    }
}

}  // namespace

cudaError_t launch_broadcast_rows(float* dst, const float* src, int32_t rows, int64_t P, int sms, cudaStream_t stream)
{
    if (rows <= 0 || P <= 0) return cudaSuccess;
    const bool vec = P % 4 == 0 && (reinterpret_cast<uintptr_t>(dst) & 15u) == 0 &&
                     (reinterpret_cast<uintptr_t>(src) & 15u) == 0;
    const int64_t count = vec ? P / 4 : P;
    int64_t grid = (count + kCopyThreads - 1) / kCopyThreads;
    const int64_t cap = (int64_t)sms * (2048 / kCopyThreads);
    if (grid > cap) grid = cap;
    if (grid < 1) grid = 1;
    if (vec)
        broadcast_rows_kernel<float4><<<(unsigned)grid, kCopyThreads, 0, stream>>>(
            reinterpret_cast<float4*>(dst), reinterpret_cast<const float4*>(src), rows, P / 4, count);
    else
        broadcast_rows_kernel<float><<<(unsigned)grid, kCopyThreads, 0, stream>>>(dst, src, rows, P, count);
    return cudaGetLastError();
}

cudaError_t launch_copy(void* dst, const void* src, int64_t bytes, int sms, cudaStream_t stream)
{
    if (bytes <= 0) return cudaSuccess;
    const int64_t n16 = bytes / 16;
    const int tail = (int)(bytes % 16);
    int64_t grid = (n16 + kCopyThreads - 1) / kCopyThreads;
    const int64_t cap = (int64_t)sms * (2048 / kCopyThreads);
    if (grid > cap) grid = cap;
    if (grid < 1) grid = 1;
    copy16_kernel<<<(unsigned)grid, kCopyThreads, 0, stream>>>(static_cast<uint4*>(dst), static_cast<const uint4*>(src),
                                                               n16, tail);
    return cudaGetLastError();
}

}  // namespace adpsgd
