// Element-type conversions between the backward's saved inputs and its
// tensor-core operands.
#include "internal.h"

#include <cuda_bf16.h>

namespace elsaa {

namespace {
__global__ void k_bf16_image(const float *__restrict__ x,
                             uint16_t *__restrict__ y, size_t n) {
    for (size_t i = (size_t)blockIdx.x * blockDim.x + threadIdx.x; i < n;
         i += (size_t)gridDim.x * blockDim.x) {
        const __nv_bfloat16 h = __float2bfloat16_rn(x[i]);
        y[i] = *reinterpret_cast<const uint16_t *>(&h);
    }
}
}  // namespace

cudaError_t launch_bf16_image(const float *x, uint16_t *y, size_t n,
                              cudaStream_t st) {
    const size_t blocks = (n + 255) / 256;
    k_bf16_image<<<(unsigned)(blocks < 1024 ? blocks : 1024), 256, 0, st>>>(
        x, y, n);
    return cudaGetLastError();
}

}  // namespace elsaa
