// Test helper: managed (unified) memory for the transfer tests, which check that a copy whose
// device side is managed memory takes the cudaMemcpyAsync route and delivers every byte.
#include <cuda_runtime.h>

extern "C" void* test_alloc_managed(size_t bytes)
{
    void* p = nullptr;
    return cudaMallocManaged(&p, bytes) == cudaSuccess ? p : nullptr;
}

extern "C" int test_free_managed(void* p) { return cudaFree(p) == cudaSuccess ? 0 : 1; }
