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

// The bf16 plane image ([H][Lg_pad][d], rows past Lg zero) and a bf16 copy
// of n4 groups of four fp32 values in one launch (both round to nearest
// even, as k_prep_planes and k_bf16_image do).
__global__ void k_planes_and_image(const float *__restrict__ w, int H,
                                   int Lg, int Lg_pad, int d,
                                   uint16_t *__restrict__ wout,
                                   const float4 *__restrict__ x,
                                   uint2 *__restrict__ y, size_t n4) {
    const size_t np = (size_t)H * Lg_pad * d;
    for (size_t i = (size_t)blockIdx.x * blockDim.x + threadIdx.x;
         i < np + n4; i += (size_t)gridDim.x * blockDim.x) {
        if (i < np) {
            const int c = (int)(i % d);
            const size_t hr = i / d;
            const int row = (int)(hr % Lg_pad), h = (int)(hr / Lg_pad);
            const float v = row < Lg ? w[((size_t)h * Lg + row) * d + c] : 0.0f;
            const __nv_bfloat16 b = __float2bfloat16_rn(v);
            wout[i] = *reinterpret_cast<const uint16_t *>(&b);
        } else {
            const float4 v = x[i - np];
            const __nv_bfloat162 lo = __floats2bfloat162_rn(v.x, v.y);
            const __nv_bfloat162 hi = __floats2bfloat162_rn(v.z, v.w);
            y[i - np] = make_uint2(*reinterpret_cast<const uint32_t *>(&lo),
                                   *reinterpret_cast<const uint32_t *>(&hi));
        }
    }
}
}  // namespace

cudaError_t launch_planes_and_image(const Plan &P, const float *w_race,
                                    uint16_t *w_bf16, const float *x,
                                    uint16_t *y, size_t n, cudaStream_t st) {
    if (n % 4 != 0 || (uintptr_t)x % 16 != 0 || (uintptr_t)y % 8 != 0)
        return cudaErrorInvalidValue;
    const size_t total = (size_t)P.H * P.Lg_pad * P.d + n / 4;
    const size_t blocks = (total + 255) / 256;
    k_planes_and_image<<<(unsigned)(blocks < 1024 ? blocks : 1024), 256, 0,
                         st>>>(w_race, P.H, P.L * P.gamma, P.Lg_pad, P.d,
                               w_bf16, reinterpret_cast<const float4 *>(x),
                               reinterpret_cast<uint2 *>(y), n / 4);
    return cudaGetLastError();
}

cudaError_t launch_bf16_image(const float *x, uint16_t *y, size_t n,
                              cudaStream_t st) {
    const size_t blocks = (n + 255) / 256;
    k_bf16_image<<<(unsigned)(blocks < 1024 ? blocks : 1024), 256, 0, st>>>(
        x, y, n);
    return cudaGetLastError();
}

}  // namespace elsaa
