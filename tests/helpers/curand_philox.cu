// Known-answer source for the Philox4x32-10 stream on the GPU: a kernel that
// calls cuRAND's curand_Philox4x32_10(counter, key) (not copied).
#include <curand_kernel.h>
#include <cstdint>

__global__ void curand_philox_kernel(const uint4* ctr, const uint2* key, uint4* out, uint64_t n) {
    const uint64_t i = static_cast<uint64_t>(blockIdx.x) * blockDim.x + threadIdx.x;
    if (i < n) out[i] = curand_Philox4x32_10(ctr[i], key[i]);
}

extern "C" int curand_philox_blocks(const void* d_ctr, const void* d_key, void* d_out, uint64_t n) {
    if (n == 0) return 0;
    curand_philox_kernel<<<static_cast<unsigned>((n + 255) / 256), 256>>>(
        static_cast<const uint4*>(d_ctr), static_cast<const uint2*>(d_key), static_cast<uint4*>(d_out), n);
    if (cudaGetLastError() != cudaSuccess) return -1;
    return cudaDeviceSynchronize() == cudaSuccess ? 0 : -2;
}
