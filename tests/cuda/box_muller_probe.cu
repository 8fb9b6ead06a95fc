// Test helper: the library's Box-Muller (noise.cuh) on chosen word pairs, so that a test can
// compare every value the generator can produce with the oracle.  Built by the test with the
// library's own arithmetic flags (no contraction, IEEE division and square root, no flush).
#include <cstdint>

#include "noise.cuh"

namespace {
__global__ void box_muller_probe_kernel(const uint32_t* wr, const uint32_t* wa, int64_t m, float* z0, float* z1)
{
    const int64_t t = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    if (t < m) adpsgd::box_muller(wr[t], wa[t], z0[t], z1[t]);
}
}  // namespace

extern "C" int box_muller_probe(const uint32_t* wr, const uint32_t* wa, int64_t m, float* z0, float* z1)
{
    if (m <= 0) return 0;
    const int64_t blocks = (m + 255) / 256;
    box_muller_probe_kernel<<<(unsigned)blocks, 256>>>(wr, wa, m, z0, z1);
    return cudaDeviceSynchronize() == cudaSuccess && cudaGetLastError() == cudaSuccess ? 0 : 1;
}
