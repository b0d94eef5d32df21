// Device helpers shared by the CUDA kernels of libelsaa.
#pragma once

#include <cuda_bf16.h>
#include <math.h>
#include <stdint.h>

#include "internal.h"

namespace elsaa {

template <typename T>
__device__ __forceinline__ float to_f32(T x);
template <>
__device__ __forceinline__ float to_f32<float>(float x) { return x; }
template <>
__device__ __forceinline__ float to_f32<__nv_bfloat16>(__nv_bfloat16 x) {
    return __bfloat162float(x);
}

template <typename T>
__device__ __forceinline__ T from_f32(float x);
template <>
__device__ __forceinline__ float from_f32<float>(float x) { return x; }
template <>
__device__ __forceinline__ __nv_bfloat16 from_f32<__nv_bfloat16>(float x) {
    return __float2bfloat16_rn(x);
}

__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
    return v;
}
__device__ __forceinline__ float warp_max(float v) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1)
        v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, o));
    return v;
}

// First fault wins; later faults keep the first record.
__device__ __forceinline__ void report(DeviceStatus *st, int code, int where,
                                       int a, int b) {
    if (st && atomicCAS(&st->code, 0, code) == 0) {
        st->where = where;
        st->info0 = a;
        st->info1 = b;
    }
}

// Rank of code c in the reflected Gray sequence k ^ (k >> 1).
__device__ __forceinline__ uint32_t gray_rank(uint32_t c) {
    uint32_t k = c;
#pragma unroll
    for (int s = 1; s < 16; s <<= 1) k ^= k >> s;
    return k;
}

// Per-bit factors of the RACE feature map. For one table with projections
// u_b = tanh(<w_b, x>), the softmax over hypercube corners v_r factorises:
// phi_r = prod_b sigmoid(2 beta u_b v_rb). Writes sp[b] = sigmoid(2 beta u_b)
// and sn[b] = sigmoid(-2 beta u_b) (both computed without cancellation).
__device__ __forceinline__ void race_bit_factors(float a, float beta,
                                                 float &sp, float &sn) {
    float t = 2.0f * beta * tanhf(a);
    float e = expf(-fabsf(t));
    float big = 1.0f / (1.0f + e);
    float small = e * big;
    sp = t >= 0.0f ? big : small;
    sn = t >= 0.0f ? small : big;
}

// Eq. (5) in its log-sum-exp form: m = exp(log d_s - log D),
// log D = LSE(log d_s, log lambda + log d_lr, log eps). mode 1: m = 1.
__device__ __forceinline__ float fusion_multiplier(float log_ds, float lam,
                                                   float dlr, float eps,
                                                   int mode) {
    if (mode == 1) return 1.0f;
    float a = log_ds;
    float b = (lam > 0.0f && dlr > 0.0f) ? logf(lam) + logf(dlr) : -INFINITY;
    float c = logf(eps);
    float mx = fmaxf(a, fmaxf(b, c));
    float s = expf(a - mx) + expf(b - mx) + expf(c - mx);
    return expf(a - (mx + logf(s)));
}

// fusion_multiplier with fast (approximate) log/exp, for the bf16 path.
__device__ __forceinline__ float fusion_multiplier_fast(float log_ds, float lam,
                                                        float dlr, float eps,
                                                        int mode) {
    if (mode == 1) return 1.0f;
    float a = log_ds;
    float b = (lam > 0.0f && dlr > 0.0f) ? __logf(lam * dlr) : -INFINITY;
    float c = __logf(eps);
    float mx = fmaxf(a, fmaxf(b, c));
    float s = __expf(a - mx) + __expf(b - mx) + __expf(c - mx);
    return __expf(a - mx) / s;
}

}  // namespace elsaa
