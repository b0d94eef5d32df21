// Token-wise gates and query-dependent lambda of the ELSAA fusion.
//
// Section 3.3 (the fusion paragraph) with the model-setup appendix: the
// gates are (g_sparse, g_lr) = sigmoid(G_theta(q_i)), G_theta a two-layer
// MLP with a SiLU hidden layer of width g and two outputs, each through its
// own sigmoid. The lambda appendix: lambda_i = max(c + sigmoid(w^T q + b),
// lambda_min). Both are per head, per query row.
//
// Tensor-core path (bf16 Q, d_h in {64, 128}): the hidden pre-activations
// and the lambda projection of a 128-query tile come out of one tcgen05 MMA
// D[128 x NG] = Q_tile [128 x d] * Wg^T, Wg = [W1; w_lambda; 0] (NG = g + 16
// rows, a bf16 image prepared per call). Each thread then owns one query
// row: it reads its NG accumulator columns from tensor memory, applies
// b1, SiLU, the 2 x g output layer, the sigmoids and the lambda rule, and
// writes (g_sparse, g_lr) and lambda_i. Persistent CTAs (two per SM) walk a
// contiguous range of tiles ordered by head, with the next two Q tiles in
// flight (TMA, 128-byte swizzle) while the current one is finished.
//
// CUDA-core path (fp32 Q, or other d_h): one thread per query row, fp32
// fused multiply-adds over the rows staged in shared memory.
#include "device_common.cuh"
#include "tc_common.cuh"
#include "tc_race.cuh"

namespace elsaa {

namespace {

using namespace tc;

constexpr int kGateThreads = 128;
constexpr int kGateMaxHidden = 128;

__device__ __forceinline__ float sigmoid_f(float x) {
    return __fdividef(1.0f, 1.0f + __expf(-x));
}
__device__ __forceinline__ float silu_f(float x) {
    return __fdividef(x, 1.0f + __expf(-x));
}

// Wg image [H][NG][d] bf16: rows [0, g) = W1[h], row g = w_lambda[h] (zero
// when absent), rows (g, NG) zero.
__global__ void k_gate_prep(const float *__restrict__ w1,
                            const float *__restrict__ w_lambda, int H, int g,
                            int NG, int d, uint16_t *__restrict__ out) {
    const long n = (long)H * NG * d;
    for (long i = blockIdx.x * (long)blockDim.x + threadIdx.x; i < n;
         i += (long)gridDim.x * blockDim.x) {
        const int c = (int)(i % d);
        const long hr = i / d;
        const int row = (int)(hr % NG), h = (int)(hr / NG);
        float x = 0.0f;
        if (row < g)
            x = w1[((long)h * g + row) * d + c];
        else if (row == g && w_lambda)
            x = w_lambda[(long)h * d + c];
        const __nv_bfloat16 b = __float2bfloat16_rn(x);
        out[i] = *reinterpret_cast<const uint16_t *>(&b);
    }
}

// Per-head small parameters staged in shared memory.
struct GateSmem {
    float b1[kGateMaxHidden];
    float w2[2][kGateMaxHidden];
    float b2[2];
    float bl, cl;
};

__device__ __forceinline__ void load_head_params(
    GateSmem &s, int h, int g, const float *b1, const float *w2,
    const float *b2, const float *b_lambda, const float *c_lambda, int tid,
    int nthreads) {
    for (int j = tid; j < g; j += nthreads) {
        s.b1[j] = b1[(long)h * g + j];
        s.w2[0][j] = w2[((long)h * 2 + 0) * g + j];
        s.w2[1][j] = w2[((long)h * 2 + 1) * g + j];
    }
    if (tid == 0) {
        s.b2[0] = b2[2 * h];
        s.b2[1] = b2[2 * h + 1];
        s.bl = b_lambda ? b_lambda[h] : 0.0f;
        s.cl = c_lambda ? c_lambda[h] : 0.0f;
    }
}

template <int D>
__global__ void __launch_bounds__(kGateThreads, 2)
    k_gate_mlp_tc(const __grid_constant__ CUtensorMap tmQ,
                  const __grid_constant__ CUtensorMap tmW,
                  const float *__restrict__ b1, const float *__restrict__ w2,
                  const float *__restrict__ b2,
                  const float *__restrict__ b_lambda,
                  const float *__restrict__ c_lambda, float lambda_min, int g,
                  int NG, uint32_t tcols, int has_lambda, int N, int H,
                  int tiles_per_head, long total_tiles,
                  float *__restrict__ gates, float *__restrict__ lam_out,
                  DeviceStatus *status) {
    extern __shared__ unsigned char smem_raw[];
    __shared__ uint64_t q_full[2], w_full, mma_done;
    __shared__ uint32_t tbase;
    __shared__ int abort_flag;
    __shared__ GateSmem ps;
    volatile int *abort = &abort_flag;
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const long t_begin = total_tiles * blockIdx.x / gridDim.x;
    const long t_end = total_tiles * (blockIdx.x + 1) / gridDim.x;
    const int ntiles = (int)(t_end - t_begin);
    constexpr uint32_t tileB = 128u * D * 2u;
    const uint32_t base = align1k(smem_u32(smem_raw));
    const uint32_t sQ0 = base, sW = base + 2 * tileB;

    if (warp == 0) tmem_alloc(&tbase, tcols);
    if (tid == 0) {
        mbar_init(&q_full[0], 1);
        mbar_init(&q_full[1], 1);
        mbar_init(&w_full, 1);
        mbar_init(&mma_done, 1);
        abort_flag = 0;
        fence_mbar_init();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = tbase;

    auto issue_q = [&](int i) {
        const long t = t_begin + i;
        const int bh = (int)(t / tiles_per_head);
        const int n0 = (int)(t - (long)bh * tiles_per_head) * 128;
        const int s = i & 1;
        mbar_expect_tx(&q_full[s], tileB);
#pragma unroll
        for (int p = 0; p < D / 64; ++p)
            tma_load_2d(sQ0 + s * tileB + p * 16384u, &tmQ, 64 * p,
                        bh * N + n0, &q_full[s]);
    };
    int issued = 0;
    if (tid == 0)
        for (; issued < 2 && issued < ntiles; ++issued) issue_q(issued);

    const uint32_t idesc = idesc_bf16(128, NG, false, false);
    int cur_h = -1, w_loads = 0, w_waits = 0;
    bool ok = true;
    int i = 0;
    for (; i < ntiles; ++i) {
        const long t = t_begin + i;
        const int bh = (int)(t / tiles_per_head);
        const int n0 = (int)(t - (long)bh * tiles_per_head) * 128;
        const int h = bh % H;
        if (h != cur_h) {
            // the previous tile's MMA and epilogue are complete: reload the
            // operand image and the small parameters of the new head
            if (tid == 0) {
                mbar_expect_tx(&w_full, (uint32_t)NG * D * 2u);
#pragma unroll
                for (int p = 0; p < D / 64; ++p)
                    tma_load_2d(sW + p * (uint32_t)NG * 128u, &tmW, 64 * p,
                                h * NG, &w_full);
                ++w_loads;
            }
            load_head_params(ps, h, g, b1, w2, b2, b_lambda, c_lambda, tid,
                             kGateThreads);
            cur_h = h;
            __syncthreads();
        }
        if (tid == 0) {
            if (w_waits < w_loads) {
                ok = mbar_wait_or_abort(&w_full, w_waits & 1, abort, status,
                                        0x6001);
                ++w_waits;
            }
            if (ok)
                ok = mbar_wait_or_abort(&q_full[i & 1], (i >> 1) & 1, abort,
                                        status, 0x6002);
            if (ok) {
                tc_fence_after();
                const uint32_t sQ = sQ0 + (i & 1) * tileB;
#pragma unroll
                for (int k = 0; k < D / 16; ++k) {
                    const uint32_t oa = (k >> 2) * 128u * 128u + (k & 3) * 32u;
                    const uint32_t ow =
                        (k >> 2) * (uint32_t)NG * 128u + (k & 3) * 32u;
                    mma_ss(tmem, smem_desc(sQ + oa, 16, 1024),
                           smem_desc(sW + ow, 16, 1024), idesc, k > 0);
                }
                mma_commit(&mma_done);
            }
        }
        if (!__syncthreads_and(ok)) break;
        ok = mbar_wait_or_abort(&mma_done, i & 1, abort, status, 0x6003);
        if (!__syncthreads_and(ok)) break;
        tc_fence_after();
        // the MMA has read Q stage i & 1: refill it with tile i + 2
        if (tid == 0 && issued < ntiles) issue_q(issued++);

        const int row = warp * 32 + lane;
        const int n = n0 + row;
        const uint32_t taddr = tmem + ((uint32_t)(warp * 32) << 16);
        float z0 = ps.b2[0], z1 = ps.b2[1];
        for (int c0 = 0; c0 < g; c0 += 16) {
            uint32_t r[16];
            tmem_ld16(taddr + c0, r);
            tmem_wait_ld();
#pragma unroll
            for (int j = 0; j < 16; ++j) {
                const float a = silu_f(__uint_as_float(r[j]) + ps.b1[c0 + j]);
                z0 = fmaf(ps.w2[0][c0 + j], a, z0);
                z1 = fmaf(ps.w2[1][c0 + j], a, z1);
            }
        }
        float lam = 0.0f;
        if (has_lambda) {
            uint32_t r[16];
            tmem_ld16(taddr + g, r);
            tmem_wait_ld();
            lam = fmaxf(ps.cl + sigmoid_f(__uint_as_float(r[0]) + ps.bl),
                        lambda_min);
        }
        if (n < N) {
            const long o = (long)bh * N + n;
            reinterpret_cast<float2 *>(gates)[o] =
                make_float2(sigmoid_f(z0), sigmoid_f(z1));
            if (has_lambda) lam_out[o] = lam;
        }
        // tensor memory and the head parameters are free for the next tile
        tc_fence_before();
        __syncthreads();
    }
    if (!ok && tid == 0) {
        // never leave with copies in flight into this CTA's shared memory
        for (int j = i; j < issued; ++j)
            mbar_wait(&q_full[j & 1], (j >> 1) & 1, nullptr, 0);
        if (w_waits < w_loads) mbar_wait(&w_full, w_waits & 1, nullptr, 0);
    }
    __syncthreads();
    if (warp == 0) tmem_dealloc(tmem, tcols);
}

// CUDA-core path: one thread per query row of a 128-row tile of one head.
template <typename T>
__global__ void __launch_bounds__(kGateThreads)
    k_gate_mlp_simt(const T *__restrict__ q, const float *__restrict__ w1,
                    const float *__restrict__ b1, const float *__restrict__ w2,
                    const float *__restrict__ b2,
                    const float *__restrict__ w_lambda,
                    const float *__restrict__ b_lambda,
                    const float *__restrict__ c_lambda, float lambda_min,
                    int g, int N, int d, int H, float *__restrict__ gates,
                    float *__restrict__ lam_out) {
    extern __shared__ float gsm[];
    __shared__ GateSmem ps;
    const int bh = blockIdx.y, h = bh % H, tid = threadIdx.x;
    const int n0 = blockIdx.x * kGateThreads;
    const int ld = d + 1;
    float *Qs = gsm;                       // [128][d + 1]
    float *Ws = Qs + kGateThreads * ld;    // [g][d]
    float *wl = Ws + g * d;                // [d]
    for (int i = tid; i < kGateThreads * d; i += kGateThreads) {
        const int rr = i / d, c = i - rr * d;
        const int n = n0 + rr;
        Qs[rr * ld + c] =
            n < N ? to_f32<T>(q[((long)bh * N + n) * d + c]) : 0.0f;
    }
    for (int i = tid; i < g * d; i += kGateThreads)
        Ws[i] = w1[(long)h * g * d + i];
    for (int i = tid; i < d; i += kGateThreads)
        wl[i] = w_lambda ? w_lambda[(long)h * d + i] : 0.0f;
    load_head_params(ps, h, g, b1, w2, b2, b_lambda, c_lambda, tid,
                     kGateThreads);
    __syncthreads();
    const int n = n0 + tid;
    if (n >= N) return;
    const float *x = Qs + tid * ld;
    float z0 = ps.b2[0], z1 = ps.b2[1];
    for (int j = 0; j < g; ++j) {
        float acc = 0.0f;
        for (int c = 0; c < d; ++c) acc = fmaf(Ws[j * d + c], x[c], acc);
        const float a = silu_f(acc + ps.b1[j]);
        z0 = fmaf(ps.w2[0][j], a, z0);
        z1 = fmaf(ps.w2[1][j], a, z1);
    }
    const long o = (long)bh * N + n;
    reinterpret_cast<float2 *>(gates)[o] =
        make_float2(sigmoid_f(z0), sigmoid_f(z1));
    if (w_lambda) {
        float acc = 0.0f;
        for (int c = 0; c < d; ++c) acc = fmaf(wl[c], x[c], acc);
        lam_out[o] = fmaxf(ps.cl + sigmoid_f(acc + ps.bl), lambda_min);
    }
}

}  // namespace

int gate_ng(int hidden) { return hidden + 16; }

bool gate_tc_supported(const Plan &P) {
    return P.dtype == ELSAA_BF16 && (P.d == 64 || P.d == 128) &&
           (long)P.BH * P.N < (1l << 31);
}

size_t gate_workspace_bytes(const Plan &P, int hidden) {
    return 256 + (size_t)P.H * gate_ng(hidden) * P.d * sizeof(uint16_t);
}

cudaError_t launch_gates(const Plan &P, const elsaa_gate_mlp &m,
                         const void *q, float *gates, float *lam_out,
                         uint16_t *w_bf16, DeviceStatus *status,
                         cudaStream_t st) {
    const int g = m.hidden, NG = gate_ng(g);
    const int has_lambda = m.w_lambda != nullptr;
    if (!gate_tc_supported(P)) {
        dim3 grid((P.N + kGateThreads - 1) / kGateThreads, P.BH);
        const size_t smem =
            sizeof(float) * ((size_t)kGateThreads * (P.d + 1) +
                             (size_t)g * P.d + P.d);
        auto launch = [&](auto kern, auto qp) {
            cudaFuncSetAttribute(kern,
                                 cudaFuncAttributeMaxDynamicSharedMemorySize,
                                 (int)smem);
            kern<<<grid, kGateThreads, smem, st>>>(
                qp, m.w1, m.b1, m.w2, m.b2, m.w_lambda, m.b_lambda,
                m.c_lambda, m.lambda_min, g, P.N, P.d, P.H, gates, lam_out);
            return cudaGetLastError();
        };
        if (P.dtype == ELSAA_FP32)
            return launch(k_gate_mlp_simt<float>, (const float *)q);
        return launch(k_gate_mlp_simt<__nv_bfloat16>,
                      (const __nv_bfloat16 *)q);
    }
    {
        const long n = (long)P.H * NG * P.d;
        const int blocks = (int)((n + 255) / 256 < 1024 ? (n + 255) / 256
                                                         : 1024);
        k_gate_prep<<<blocks, 256, 0, st>>>(m.w1, m.w_lambda, P.H, g, NG, P.d,
                                            w_bf16);
        cudaError_t e = cudaGetLastError();
        if (e != cudaSuccess) return e;
    }
    CUtensorMap tmQ, tmW;
    cudaError_t e = make_tma_map_bf16(&tmQ, q, (uint64_t)P.BH * P.N, P.d, 128);
    if (e == cudaSuccess)
        e = make_tma_map_bf16(&tmW, w_bf16, (uint64_t)P.H * NG, P.d,
                              (uint32_t)NG);
    if (e != cudaSuccess) return e;
    const uint32_t tcols = NG <= 32 ? 32u : NG <= 64 ? 64u : NG <= 128 ? 128u
                                                                     : 256u;
    const int tiles_per_head = (P.N + 127) / 128;
    const long total = (long)tiles_per_head * P.BH;
    int dev = 0, sms = 148;
    if (cudaGetDevice(&dev) == cudaSuccess)
        cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    const long slots = 2l * sms;
    const int grid = (int)(total < slots ? total : slots);
    const size_t smem = 1024 + 2 * (size_t)128 * P.d * 2 +
                        (size_t)NG * P.d * 2;
    auto launch = [&](auto kern) {
        cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             (int)smem);
        kern<<<grid, kGateThreads, smem, st>>>(
            tmQ, tmW, m.b1, m.w2, m.b2, m.b_lambda, m.c_lambda, m.lambda_min,
            g, NG, tcols, has_lambda, P.N, P.H, tiles_per_head, total, gates,
            lam_out, status);
        return cudaGetLastError();
    };
    return P.d == 64 ? launch(k_gate_mlp_tc<64>) : launch(k_gate_mlp_tc<128>);
}

}  // namespace elsaa
