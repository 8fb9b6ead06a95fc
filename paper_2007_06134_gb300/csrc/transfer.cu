// transfer.cu -- host <-> device copies carried out by the SMs: a grid-stride copy kernel that
// reads or writes page-locked host memory through its mapped device address.  The copy engines
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

}  // namespace

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
