// Token-wise gates and query-dependent lambda of the ELSAA fusion.
//
// Section 3.3 (the fusion paragraph) with Appendix D (experiment
// hyperparameters): the gates are (g_sparse, g_lr) = sigmoid(G_theta(q_i)),
// G_theta a two-layer MLP with a SiLU hidden layer of width g and two
// outputs, each through its own sigmoid. Appendix D, input-dependent
// lambda: lambda_i = max(c + sigmoid(w^T q + b), lambda_min). Both are per
// head, per query row.
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

// sigmoid(x) = 1 / (1 + 2^(-x log2 e)) from the hardware base-2
// exponential and reciprocal (both approximate to about 2^-22 relative).
// Tails: x -> -inf gives 2^(+inf) = inf and 1 / inf = 0; x -> +inf gives 1.
__device__ __forceinline__ float ex2_ftz(float x) {
    float y;
    asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
    return y;
}
__device__ __forceinline__ float rcp_ftz(float x) {
    float y;
    asm("rcp.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
    return y;
}
constexpr float kNegLog2e = -1.4426950408889634f;
__device__ __forceinline__ float sigmoid_f(float x) {
    return rcp_ftz(1.0f + ex2_ftz(x * kNegLog2e));
}
// SiLU(x) = x sigmoid(x)
__device__ __forceinline__ float silu_f(float x) { return x * sigmoid_f(x); }

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
struct __align__(16) GateSmem {
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

// Warp roles of k_gate_mlp_tc.
constexpr int kGateWsThreads = 320;  // producer, MMA, 8 epilogue warps
constexpr int kGateEpiThreads = 256;

template <int D>
constexpr int gate_stages() { return D == 64 ? 8 : 4; }

// Tensor-core gate kernel, warp-specialised:
//   warp 0      TMA producer: Q tiles into a ring of gate_stages<D>()
//               stages (128-byte swizzle panels).
//   warp 1      allocates all 512 tensor-memory columns as nacc = 4 (or 2
//               when g > 112) accumulators; lane 0 issues the MMAs of tile
//               i into accumulator i mod nacc (and reloads the operand image
//               Wg when the head changes, after its earlier MMAs are done).
//   warps 2-9   epilogue, two groups of four: group G (warps 2-5, 6-9)
//               finishes the tiles i = G (mod 2); warp e
//               reads TMEM lanes 32 (e mod 4) .. 32 (e mod 4) + 31 and each
//               thread evaluates the whole MLP of one query row, so the
//               groups never wait for each other.
template <int D>
__global__ void __launch_bounds__(kGateWsThreads, 1)
    k_gate_mlp_tc(const __grid_constant__ CUtensorMap tmQ,
                  const __grid_constant__ CUtensorMap tmW,
                  const float *__restrict__ b1, const float *__restrict__ w2,
                  const float *__restrict__ b2,
                  const float *__restrict__ b_lambda,
                  const float *__restrict__ c_lambda, float lambda_min, int g,
                  int NG, uint32_t acc_cols, int has_lambda, int N, int H,
                  int tiles_per_head, long total_tiles,
                  float *__restrict__ gates, float *__restrict__ lam_out,
                  DeviceStatus *status) {
    constexpr int S = gate_stages<D>();
    extern __shared__ unsigned char smem_raw[];
    __shared__ uint64_t full[S], empty[S], acc_full[4], acc_empty[4];
    __shared__ uint64_t w_full, drain;
    __shared__ uint32_t tbase;
    __shared__ int abort_flag;
    volatile int *abort = &abort_flag;
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const long t_begin = total_tiles * blockIdx.x / gridDim.x;
    const long t_end = total_tiles * (blockIdx.x + 1) / gridDim.x;
    const int ntiles = (int)(t_end - t_begin);
    constexpr uint32_t tileB = 128u * D * 2u;
    const uint32_t base = align1k(smem_u32(smem_raw));
    const uint32_t sW = base + S * tileB;

    // nacc accumulators of acc_cols columns fill the 512 TMEM columns
    const int nacc = (int)(512u / acc_cols) < 4 ? (int)(512u / acc_cols) : 4;
    if (warp == 1) tmem_alloc(&tbase, 512);
    if (tid == 0) {
        for (int s = 0; s < S; ++s) {
            mbar_init(&full[s], 1);
            mbar_init(&empty[s], 1);
        }
        for (int a = 0; a < 4; ++a) {
            mbar_init(&acc_full[a], 1);
            mbar_init(&acc_empty[a], 4);  // the four warps of group a
        }
        mbar_init(&w_full, 1);
        mbar_init(&drain, 1);
        abort_flag = 0;
        fence_mbar_init();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = tbase;
    auto tile_of = [&](int i, int &bh, int &n0) {
        const long t = t_begin + i;
        bh = (int)(t / tiles_per_head);
        n0 = (int)(t - (long)bh * tiles_per_head) * 128;
    };

    if (warp == 0) {
        // ---------------------------------------------------- TMA producer
        if (lane == 0) {
            int i = 0;
            for (; i < ntiles; ++i) {
                const int s = i % S;
                if (i >= S && !mbar_wait_or_abort(&empty[s],
                                                  ((i / S) - 1) & 1, abort,
                                                  status, 0x6101))
                    break;
                int bh, n0;
                tile_of(i, bh, n0);
                mbar_expect_tx(&full[s], tileB);
#pragma unroll
                for (int p = 0; p < D / 64; ++p)
                    tma_load_2d(base + s * tileB + p * 16384u, &tmQ, 64 * p,
                                bh * N + n0, &full[s]);
            }
            // the last load issued into every stage has landed
            for (int s = 0; s < S; ++s) {
                const int last = i - 1 - (((i - 1 - s) % S) + S) % S;
                if (last >= 0 && last < i)
                    mbar_wait(&full[s], (last / S) & 1, status, 0x6107);
            }
        }
    } else if (warp == 1) {
        // ------------------------------------------------------------ MMA
        if (lane == 0) {
            const uint32_t idesc = idesc_bf16(128, NG, false, false);
            int cur_h = -1, drains = 0, wl = 0;
            bool ok = true;
            for (int i = 0; i < ntiles && ok; ++i) {
                int bh, n0;
                tile_of(i, bh, n0);
                const int h = bh % H;
                if (h != cur_h) {
                    if (i > 0) {  // earlier MMAs still read the old image
                        mma_commit(&drain);
                        ok = mbar_wait_or_abort(&drain, drains & 1, abort,
                                                status, 0x6102);
                        ++drains;
                        if (!ok) break;
                    }
                    mbar_expect_tx(&w_full, (uint32_t)NG * D * 2u);
#pragma unroll
                    for (int p = 0; p < D / 64; ++p)
                        tma_load_2d(sW + p * (uint32_t)NG * 128u, &tmW,
                                    64 * p, h * NG, &w_full);
                    ok = mbar_wait_or_abort(&w_full, wl & 1, abort, status,
                                            0x6103);
                    ++wl;
                    if (!ok) break;
                    cur_h = h;
                }
                const int s = i % S, a = i % nacc;
                ok = mbar_wait_or_abort(&full[s], (i / S) & 1, abort, status,
                                        0x6104);
                if (ok && i >= nacc)
                    ok = mbar_wait_or_abort(&acc_empty[a],
                                            ((i / nacc) - 1) & 1, abort,
                                            status, 0x6105);
                if (!ok) break;
                tc_fence_after();
                const uint32_t sQ = base + s * tileB;
                const uint32_t dst = tmem + a * acc_cols;
#pragma unroll
                for (int k = 0; k < D / 16; ++k) {
                    const uint32_t oa = (k >> 2) * 128u * 128u + (k & 3) * 32u;
                    const uint32_t ow =
                        (k >> 2) * (uint32_t)NG * 128u + (k & 3) * 32u;
                    mma_ss(dst, smem_desc(sQ + oa, 16, 1024),
                           smem_desc(sW + ow, 16, 1024), idesc, k > 0);
                }
                mma_commit(&empty[s]);
                mma_commit(&acc_full[a]);
            }
            // no MMA may still be writing tensor memory or reading the
            // image when the CTA ends
            mma_commit(&drain);
            mbar_wait(&drain, drains & 1, status, 0x6108);
        }
        __syncwarp();
    } else {
        // ------------------------------------------------------- epilogue
        // group G = (warp - 2) / 4 finishes the tiles i = G (mod 2), which
        // the MMA warp puts in accumulator i mod nacc; thread = one row
        const int grp = (warp - 2) >> 2;
        const int quarter = warp & 3;
        const int row = quarter * 32 + lane;
        const uint32_t lane_off = (uint32_t)(quarter * 32) << 16;
        for (int i = grp; i < ntiles; i += 2) {
            const int a = i % nacc;
            const uint32_t taddr = tmem + a * acc_cols + lane_off;
            int bh, n0;
            tile_of(i, bh, n0);
            const int h = bh % H;
            // per-head parameters straight from global memory (L1-cached,
            // one address per warp): no barrier between the warps
            const float4 *pb4 = reinterpret_cast<const float4 *>(b1 + (long)h * g);
            const float4 *pw0 =
                reinterpret_cast<const float4 *>(w2 + (long)h * 2 * g);
            const float4 *pw1 =
                reinterpret_cast<const float4 *>(w2 + ((long)h * 2 + 1) * g);
            if (!mbar_wait_or_abort(&acc_full[a], (i / nacc) & 1, abort,
                                    status, 0x6106))
                break;
            tc_fence_after();
            // four partial sums per output keep the FMA chains short
            float z0[4] = {__ldg(b2 + 2 * h), 0.0f, 0.0f, 0.0f};
            float z1[4] = {__ldg(b2 + 2 * h + 1), 0.0f, 0.0f, 0.0f};
            for (int c0 = 0; c0 < g; c0 += 16) {
                uint32_t r[16];
                tmem_ld16(taddr + c0, r);
                tmem_wait_ld();
#pragma unroll
                for (int j4 = 0; j4 < 4; ++j4) {
                    const float4 bb = __ldg(pb4 + c0 / 4 + j4);
                    const float4 u0 = __ldg(pw0 + c0 / 4 + j4);
                    const float4 u1 = __ldg(pw1 + c0 / 4 + j4);
                    const float bv[4] = {bb.x, bb.y, bb.z, bb.w};
                    const float v0[4] = {u0.x, u0.y, u0.z, u0.w};
                    const float v1[4] = {u1.x, u1.y, u1.z, u1.w};
#pragma unroll
                    for (int j = 0; j < 4; ++j) {
                        const float act =
                            silu_f(__uint_as_float(r[4 * j4 + j]) + bv[j]);
                        z0[j] = fmaf(v0[j], act, z0[j]);
                        z1[j] = fmaf(v1[j], act, z1[j]);
                    }
                }
            }
            const float s0 = (z0[0] + z0[1]) + (z0[2] + z0[3]);
            const float s1 = (z1[0] + z1[1]) + (z1[2] + z1[3]);
            float lam = 0.0f;
            if (has_lambda) {
                uint32_t r[16];
                tmem_ld16(taddr + g, r);
                tmem_wait_ld();
                lam = fmaxf(__ldg(c_lambda + h) +
                                sigmoid_f(__uint_as_float(r[0]) +
                                          __ldg(b_lambda + h)),
                            lambda_min);
            }
            // accumulator a is free for tile i + nacc
            tc_fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive(&acc_empty[a]);
            if (n0 + row < N) {
                const long o = (long)bh * N + n0 + row;
                reinterpret_cast<float2 *>(gates)[o] =
                    make_float2(sigmoid_f(s0), sigmoid_f(s1));
                if (has_lambda) lam_out[o] = lam;
            }
        }
    }
    __syncthreads();
    if (warp == 1) tmem_dealloc(tmem, 512);
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
    const uint32_t acc_cols = NG <= 32 ? 32u : NG <= 64 ? 64u
                              : NG <= 128 ? 128u : 256u;
    const int tiles_per_head = (P.N + 127) / 128;
    const long total = (long)tiles_per_head * P.BH;
    int dev = 0, sms = 148;
    if (cudaGetDevice(&dev) == cudaSuccess)
        cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    const int grid = (int)(total < sms ? total : sms);
    auto launch = [&](auto kern, int stages) {
        const size_t smem = 1024 + (size_t)stages * 128 * P.d * 2 +
                            (size_t)NG * P.d * 2;
        cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             (int)smem);
        kern<<<grid, kGateWsThreads, smem, st>>>(
            tmQ, tmW, m.b1, m.w2, m.b2, m.b_lambda, m.c_lambda, m.lambda_min,
            g, NG, acc_cols, has_lambda, P.N, P.H, tiles_per_head, total,
            gates, lam_out, status);
        return cudaGetLastError();
    };
    return P.d == 64 ? launch(k_gate_mlp_tc<64>, gate_stages<64>())
                     : launch(k_gate_mlp_tc<128>, gate_stages<128>());
}

}  // namespace elsaa
