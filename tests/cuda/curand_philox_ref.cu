// Test-only reference: Philox4x32-10 blocks from cuRAND's device API, to pin both the oracle's
// and the library's Philox against an independent implementation.  For each (q, i) it writes
//   raw[t]  = curand_Philox4x32_10(counter (q, i, k, tag), key (seed lo, seed hi))
//   api[t]  = curand4() after curand_init(seed, subsequence = k + 2^32 tag,
//             offset = 4 (q + 2^32 i)), i.e. the same counter reached through the documented API.
#include <cuda_runtime.h>
#include <curand_kernel.h>

__global__ void ref_kernel(unsigned long long seed, unsigned tag, int n, long long nq, unsigned k, uint4* raw,
                           uint4* api)
{
    const long long t = (long long)blockIdx.x * blockDim.x + threadIdx.x;
    if (t >= (long long)n * nq) return;
    const unsigned i = (unsigned)(t / nq);
    const unsigned q = (unsigned)(t % nq);
    raw[t] = curand_Philox4x32_10(make_uint4(q, i, k, tag),
                                  make_uint2((unsigned)(seed & 0xFFFFFFFFull), (unsigned)(seed >> 32)));
    curandStatePhilox4_32_10_t st;
    const unsigned long long subsequence = (unsigned long long)k | ((unsigned long long)tag << 32);
    const unsigned long long offset = 4ull * ((unsigned long long)q | ((unsigned long long)i << 32));
    curand_init(seed, subsequence, offset, &st);
    api[t] = curand4(&st);
}

extern "C" int curand_ref_fill(unsigned long long seed, unsigned tag, int n, long long nq, unsigned k, void* raw,
                               void* api)
{
    const long long total = (long long)n * nq;
    const int threads = 256;
    const long long blocks = (total + threads - 1) / threads;
    if (blocks > 0)
        ref_kernel<<<(unsigned)blocks, threads>>>(seed, tag, n, nq, k, static_cast<uint4*>(raw),
                                                  static_cast<uint4*>(api));
    cudaError_t e = cudaGetLastError();
    if (e == cudaSuccess) e = cudaDeviceSynchronize();
    return (int)e;
}
