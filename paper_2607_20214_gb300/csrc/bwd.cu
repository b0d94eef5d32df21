// Backward pass of the ELSAA operator, CUDA cores, fp32 (all dtypes).
//
// The derivative of the forward definitions: sortLSH block attention
// (Algorithm "sortLSH Sparse Exact Attention Branch", block step), the RACE
// summaries and readout (Algorithm "RACE Low-Rank Attention Branch") and the
// fusion of Eq. (5)-(6). The hash and the sort carry no gradient; the
// forward's permutations are inputs. Launches, in order:
//   k_race_partial / k_race_reduce    A, B again (as in the forward)
//   k_bwd_block                       one CTA per (sorted block, head):
//                                     the block-local sparse gradient
//                                     (dQ, dK, dV of the block: every key
//                                     belongs to exactly one block, so no
//                                     atomics), the query side of RACE
//                                     (dQ through phi, tanh and W), and
//                                     gNum / L, gDen / L per query
//   k_race_partial (weighted) / reduce  gB = sum_i phi(Q_i) gNum_i^T / L,
//                                     gA = sum_i phi(Q_i) gDen_i / L
//   k_bwd_keys                        per key: dV += phi(K_j)^T gB,
//                                     dK += (gB V_j + gA) back through phi
//
// Per-query scalars stay in the log domain where the forward does:
// log d_s = M + log l, log D = LSE(log d_s, log(lambda Den + eps)),
// m = exp(log d_s - log D), and e^M / D = m / l, so nothing overflows for
// large scores.
#include "device_common.cuh"

namespace elsaa {

namespace {

constexpr int kBwdThreads = 256;
constexpr int kKeyThreads = 256;
constexpr int kBwdMaxB = 1024;
constexpr int kKeyTile = 32;

// log(exp(a) + exp(b)), b may be -inf
__device__ __forceinline__ float lse2(float a, float b) {
    const float mx = fmaxf(a, b);
    if (mx == -INFINITY) return -INFINITY;
    return mx + logf(expf(a - mx) + expf(b - mx));
}

// C = A B on 4 x 4 register tiles spread over the CTA's threads. Element
// (m, k) of A is A[m * am + k * ak] and (k, n) of B is B[k * bk + n * bn]
// (shared or global memory: transposes are stride swaps); epi(m, n, value)
// receives every element of C with m < M, n < N.
template <int TM = 4, typename Epi>
__device__ __forceinline__ void tile_gemm(int M, int N, int K,
                                          const float *A, int am, int ak,
                                          const float *B, int bk, int bn,
                                          Epi epi) {
    const int tn = (N + 3) >> 2, tm = (M + TM - 1) / TM;
    for (int t = threadIdx.x; t < tm * tn; t += blockDim.x) {
        const int m0 = (t / tn) * TM, n0 = (t % tn) * 4;
        float c[TM][4];
#pragma unroll
        for (int u = 0; u < TM; ++u)
#pragma unroll
            for (int w = 0; w < 4; ++w) c[u][w] = 0.f;
        for (int k = 0; k < K; ++k) {
            float a[TM], bb[4];
#pragma unroll
            for (int u = 0; u < TM; ++u)
                a[u] = (m0 + u < M) ? A[(m0 + u) * am + k * ak] : 0.f;
#pragma unroll
            for (int w = 0; w < 4; ++w)
                bb[w] = (n0 + w < N) ? B[k * bk + (n0 + w) * bn] : 0.f;
#pragma unroll
            for (int u = 0; u < TM; ++u)
#pragma unroll
                for (int w = 0; w < 4; ++w) c[u][w] = fmaf(a[u], bb[w], c[u][w]);
        }
#pragma unroll
        for (int u = 0; u < TM; ++u)
#pragma unroll
            for (int w = 0; w < 4; ++w)
                if (m0 + u < M && n0 + w < N) epi(m0 + u, n0 + w, c[u][w]);
    }
}

// u_b = tanh(<w_b, x>) for the G planes of table l, and phi_r of that table
// (product form of the softmax over corners, v_rb = +1 if bit b of r set).
template <int kMaxG>
__device__ __forceinline__ void table_features(const float *w, const float *x,
                                               int d, int G, float beta,
                                               float *u, float *phi) {
    float sp[kMaxG], sn[kMaxG];
    for (int bb = 0; bb < G; ++bb) {
        float a = 0.f;
        for (int e = 0; e < d; ++e) a = fmaf(w[bb * d + e], x[e], a);
        u[bb] = tanhf(a);
        race_bit_factors(a, beta, sp[bb], sn[bb]);
    }
    const int R = 1 << G;
    for (int rr = 0; rr < R; ++rr) {
        float pr = 1.f;
        for (int bb = 0; bb < G; ++bb) pr *= ((rr >> bb) & 1) ? sp[bb] : sn[bb];
        phi[rr] = pr;
    }
}

// dL/d(W x) of one table from dL/dphi: through the softmax over corners
// (ga_r = phi_r (gphi_r - sum phi gphi)), beta u^T v_r and tanh. Overwrites
// u[b] with (1 - u_b^2) * beta * sum_r v_rb ga_r.
__device__ __forceinline__ void table_backward(const float *phi,
                                               const float *gphi, int G,
                                               float beta, float *u) {
    const int R = 1 << G;
    float s = 0.f;
    for (int rr = 0; rr < R; ++rr) s = fmaf(phi[rr], gphi[rr], s);
    for (int bb = 0; bb < G; ++bb) {
        float gu = 0.f;
        for (int rr = 0; rr < R; ++rr) {
            const float ga = phi[rr] * (gphi[rr] - s);
            gu += ((rr >> bb) & 1) ? ga : -ga;
        }
        u[bb] = (1.f - u[bb] * u[bb]) * beta * gu;
    }
}

template <typename T>
__global__ void __launch_bounds__(kBwdThreads)
    k_bwd_block(const T *__restrict__ qx, const T *__restrict__ kx,
                const T *__restrict__ vx, const T *__restrict__ gx,
                const float *__restrict__ w_race, const float *__restrict__ Ag,
                const float *__restrict__ Bg,
                const int32_t *__restrict__ perm_q,
                const int32_t *__restrict__ perm_k,
                const float *__restrict__ lambda_tok,
                const float *__restrict__ gates, int N, int d, int H, int b,
                int L, int G, float beta, float eps, float scale,
                float lambda, int mode, float *__restrict__ dq,
                float *__restrict__ dk, float *__restrict__ dv,
                float *__restrict__ d_gates, float *__restrict__ d_lambda,
                float *__restrict__ gnum, float *__restrict__ gden,
                DeviceStatus *status) {
    extern __shared__ float sm[];
    __shared__ int qi[kBwdMaxB], ki[kBwdMaxB];
    const int t = blockIdx.x, bh = blockIdx.y, h = bh % H, tid = threadIdx.x;
    const int R = 1 << G, r = L * R, LG = L * G;
    const int dp = d + 1, bp = b + 1;
    float *Qs = sm;              // [b][d+1] queries of the block
    float *Ks = Qs + b * dp;     // keys of the block
    float *Vs = Ks + b * dp;     // values of the block
    float *Gs = Vs + b * dp;     // dO rows of the queries
    float *Es = Gs + b * dp;     // [b][b+1] scores -> exp(z - M) -> dZ
    float *Xs = Es + b * bp;     // [b][d+1] O_s, then gN_s e^M
    float *Ys = Xs + b * dp;     // [b][d+1] Num, then gNum
    float *Ph = Ys + b * dp;     // [b][r] phi(Q_i)
    float *Gp = Ph + b * r;      // [b][r] dL/dphi(Q_i)
    float *Us = Gp + b * r;      // [b][L*G] u, then dL/d(W q)
    float *sM = Us + b * LG;     // per-query scalars [b] each
    float *sl = sM + b, *sDen = sl + b, *sfN = sDen + b, *sgdsE = sfN + b;
    float *sfNum = sgdsE + b, *sgDen = sfNum + b;

    const size_t base = (size_t)bh * N;
    for (int i = tid; i < b; i += kBwdThreads) {
        // entries outside [0, N) are recorded and read as row 0
        int a = perm_q[base + (size_t)t * b + i];
        int c = perm_k[base + (size_t)t * b + i];
        if (a < 0 || a >= N) {
            report(status, kDevPermRange, 12, bh, a);
            a = 0;
        }
        if (c < 0 || c >= N) {
            report(status, kDevPermRange, 13, bh, c);
            c = 0;
        }
        qi[i] = a;
        ki[i] = c;
    }
    __syncthreads();
    for (int x = tid; x < b * d; x += kBwdThreads) {
        const int i = x / d, e = x - i * d;
        Qs[i * dp + e] = to_f32<T>(qx[(base + qi[i]) * d + e]);
        Gs[i * dp + e] = to_f32<T>(gx[(base + qi[i]) * d + e]);
        Ks[i * dp + e] = to_f32<T>(kx[(base + ki[i]) * d + e]);
        Vs[i * dp + e] = to_f32<T>(vx[(base + ki[i]) * d + e]);
    }
    __syncthreads();
    // z_ij = scale <Q_i, K_j>
    tile_gemm(b, b, d, Qs, dp, 1, Ks, 1, dp,
              [&](int i, int j, float v) { Es[i * bp + j] = scale * v; });
    __syncthreads();
    for (int i = tid; i < b; i += kBwdThreads) {
        float mx = -INFINITY;
        for (int j = 0; j < b; ++j) mx = fmaxf(mx, Es[i * bp + j]);
        float l = 0.f;
        for (int j = 0; j < b; ++j) {
            const float e = expf(Es[i * bp + j] - mx);
            Es[i * bp + j] = e;
            l += e;
        }
        sM[i] = mx;
        sl[i] = l;
        sfN[i] = 1.f / (l + eps * expf(-mx));  // (d_s + eps)^-1 e^M
    }
    __syncthreads();
    // O_s = sum_j e^(z - M) V_j / (l + eps e^-M)
    tile_gemm(b, d, b, Es, bp, 1, Vs, dp, 1, [&](int i, int e, float v) {
        Xs[i * dp + e] = v * sfN[i];
    });
    // RACE features of the queries
    for (int x = tid; x < b * L; x += kBwdThreads) {
        const int i = x / L, l = x - i * L;
        table_features<6>(w_race + ((size_t)h * L + l) * G * d, Qs + i * dp, d,
                          G, beta, Us + i * LG + l * G, Ph + i * r + l * R);
    }
    __syncthreads();
    const float *Bh_ = Bg + (size_t)bh * r * d;
    const float *Ah = Ag + (size_t)bh * r;
    // Num = (1/L) sum phi B, Den = (1/L) sum phi . A
    tile_gemm(b, d, r, Ph, r, 1, Bh_, d, 1, [&](int i, int e, float v) {
        Ys[i * dp + e] = v / (float)L;
    });
    for (int i = tid; i < b; i += kBwdThreads) {
        float a = 0.f;
        for (int rr = 0; rr < r; ++rr) a = fmaf(Ph[i * r + rr], Ah[rr], a);
        sDen[i] = a / (float)L;
    }
    __syncthreads();
    // per-query scalars: Eq. (6) then Eq. (5) backward
    for (int i = tid; i < b; i += kBwdThreads) {
        const size_t tok = base + qi[i];
        const float lam = lambda_tok ? lambda_tok[tok] : lambda;
        const float gs = gates ? gates[2 * tok] : 1.f;
        const float gl = gates ? gates[2 * tok + 1] : 1.f;
        const float M = sM[i], l = sl[i], Den = sDen[i];
        const float lsE = l + eps * expf(-M);  // (d_s + eps) e^-M
        float GOs = 0.f, GOlr = 0.f;
        for (int e = 0; e < d; ++e) {
            GOs = fmaf(Gs[i * dp + e], Xs[i * dp + e], GOs);
            GOlr = fmaf(Gs[i * dp + e], Ys[i * dp + e], GOlr);
        }
        GOlr /= (Den + eps);
        const float logds = M + logf(l);
        const float c = lam * Den + eps;
        const float logD = c > 0.f ? lse2(logds, logf(c)) : logds;
        const float m = mode == 1 ? 1.f : expf(logds - logD);
        const float invD = expf(-logD);
        const float dm = mode == 1 ? 0.f : gs * GOs;
        // gN_s e^M = g_s m G / lsE; e^M dL/dd_s = -(g_s m G.O_s) / lsE
        //   + dm (c / D) (e^M / D), with e^M / D = m / l
        sfN[i] = gs * m / lsE;
        sgdsE[i] = -(gs * m * GOs) / lsE + dm * (c * invD) * (m / l);
        // RACE: gNum = g_lr G / (Den + eps); dL/dDen = -(g_lr G.O_lr) /
        //   (Den + eps) - dm lambda d_s / D^2, with d_s / D = m
        sfNum[i] = gl / (Den + eps);
        sgDen[i] = -(gl * GOlr) / (Den + eps) - dm * lam * m * invD;
        if (d_gates) {
            d_gates[2 * tok] = m * GOs;
            d_gates[2 * tok + 1] = GOlr;
        }
        if (d_lambda) d_lambda[tok] = -dm * m * Den * invD;
    }
    __syncthreads();
    for (int x = tid; x < b * d; x += kBwdThreads) {
        const int i = x / d, e = x - i * d;
        Xs[i * dp + e] = sfN[i] * Gs[i * dp + e];    // gN_s e^M
        Ys[i * dp + e] = sfNum[i] * Gs[i * dp + e];  // gNum
    }
    __syncthreads();
    // dV_j (sparse) = sum_i e^(z_ij - M_i) gN_s,i e^(M_i)
    tile_gemm(b, d, b, Es, 1, bp, Xs, dp, 1, [&](int j, int e, float v) {
        dv[(base + ki[j]) * d + e] = v;
    });
    __syncthreads();
    // dZ_ij = e^(z - M) (gN_s e^M . V_j + e^M dL/dd_s)
    tile_gemm(b, b, d, Xs, dp, 1, Vs, 1, dp, [&](int i, int j, float v) {
        Es[i * bp + j] *= (v + sgdsE[i]);
    });
    // dL/dphi(Q_i) = (B gNum_i + A dL/dDen_i) / L
    tile_gemm(b, r, d, Ys, dp, 1, Bh_, 1, d, [&](int i, int rr, float v) {
        Gp[i * r + rr] = (v + Ah[rr] * sgDen[i]) / (float)L;
    });
    __syncthreads();
    for (int x = tid; x < b * L; x += kBwdThreads) {
        const int i = x / L, l = x - i * L;
        table_backward(Ph + i * r + l * R, Gp + i * r + l * R, G, beta,
                       Us + i * LG + l * G);
    }
    // dK_j (sparse) = scale sum_i dZ_ij Q_i
    tile_gemm(b, d, b, Es, 1, bp, Qs, dp, 1, [&](int j, int e, float v) {
        dk[(base + ki[j]) * d + e] = scale * v;
    });
    // dQ_i = scale sum_j dZ_ij K_j (into Xs, free after dZ)
    tile_gemm(b, d, b, Es, bp, 1, Ks, dp, 1, [&](int i, int e, float v) {
        Xs[i * dp + e] = scale * v;
    });
    __syncthreads();
    // ... + sum_(l,b) W_lb dL/d(W q)_lb
    const float *wh = w_race + (size_t)h * LG * d;
    tile_gemm(b, d, LG, Us, LG, 1, wh, d, 1, [&](int i, int e, float v) {
        const size_t row = base + qi[i];
        dq[row * d + e] = Xs[i * dp + e] + v;
        gnum[row * d + e] = Ys[i * dp + e] / (float)L;
    });
    for (int i = tid; i < b; i += kBwdThreads)
        gden[base + qi[i]] = sgDen[i] / (float)L;
}

// Key side of RACE: dV_j += phi(K_j)^T gB, dL/dphi(K_j) = gB V_j + gA, then
// back through the features into dK_j. Grid (ceil(N / 32), B*H).
template <typename T>
__global__ void __launch_bounds__(kKeyThreads)
    k_bwd_keys(const T *__restrict__ kx, const T *__restrict__ vx,
               const float *__restrict__ w_race, const float *__restrict__ gA,
               const float *__restrict__ gB, int N, int d, int H, int L,
               int G, float beta, float *__restrict__ dk,
               float *__restrict__ dv) {
    extern __shared__ float sm[];
    const int j0 = blockIdx.x * kKeyTile, bh = blockIdx.y, h = bh % H;
    const int tid = threadIdx.x;
    const int R = 1 << G, r = L * R, LG = L * G, dp = d + 1;
    const int nk = min(kKeyTile, N - j0);
    float *Ks = sm;                  // [32][d+1]
    float *Vs = Ks + kKeyTile * dp;  // [32][d+1]
    float *Ph = Vs + kKeyTile * dp;  // [32][r]
    float *Gp = Ph + kKeyTile * r;   // [32][r]
    float *Us = Gp + kKeyTile * r;   // [32][L*G]
    const size_t base = (size_t)bh * N + j0;
    for (int x = tid; x < nk * d; x += kKeyThreads) {
        const int j = x / d, e = x - j * d;
        Ks[j * dp + e] = to_f32<T>(kx[(base + j) * d + e]);
        Vs[j * dp + e] = to_f32<T>(vx[(base + j) * d + e]);
    }
    __syncthreads();
    for (int x = tid; x < nk * L; x += kKeyThreads) {
        const int j = x / L, l = x - j * L;
        table_features<6>(w_race + ((size_t)h * L + l) * G * d, Ks + j * dp, d,
                          G, beta, Us + j * LG + l * G, Ph + j * r + l * R);
    }
    __syncthreads();
    const float *gBh = gB + (size_t)bh * r * d;
    const float *gAh = gA + (size_t)bh * r;
    tile_gemm(nk, d, r, Ph, r, 1, gBh, d, 1, [&](int j, int e, float v) {
        dv[(base + j) * d + e] += v;
    });
    tile_gemm(nk, r, d, Vs, dp, 1, gBh, 1, d, [&](int j, int rr, float v) {
        Gp[j * r + rr] = v + gAh[rr];
    });
    __syncthreads();
    for (int x = tid; x < nk * L; x += kKeyThreads) {
        const int j = x / L, l = x - j * L;
        table_backward(Ph + j * r + l * R, Gp + j * r + l * R, G, beta,
                       Us + j * LG + l * G);
    }
    __syncthreads();
    const float *wh = w_race + (size_t)h * LG * d;
    tile_gemm(nk, d, LG, Us, LG, 1, wh, d, 1, [&](int j, int e, float v) {
        dk[(base + j) * d + e] += v;
    });
}

}  // namespace

size_t bwd_block_smem(const Plan &P) {
    const size_t b = P.b, d = P.d;
    return sizeof(float) * (6 * b * (d + 1) + b * (b + 1) + 2 * b * P.r +
                            b * P.L * P.gamma + 7 * b);
}

size_t bwd_keys_smem(const Plan &P) {
    return sizeof(float) * ((size_t)kKeyTile * (2 * (P.d + 1) + 2 * P.r +
                                                 P.L * P.gamma));
}

bool bwd_supported(const Plan &P) {
    return P.b <= kBwdMaxB && P.gamma <= 6 &&
           bwd_block_smem(P) + 2 * sizeof(int) * kBwdMaxB <= 227 * 1024 &&
           bwd_keys_smem(P) <= 227 * 1024;
}

cudaError_t launch_bwd_block(const Plan &P, const void *q, const void *k,
                             const void *v, const void *d_o,
                             const float *w_race, const float *A,
                             const float *Bm, const int32_t *perm_q,
                             const int32_t *perm_k, const float *lambda_tok,
                             const float *gates, float *dq, float *dk,
                             float *dv, float *d_gates, float *d_lambda,
                             float *gnum, float *gden, DeviceStatus *status,
                             cudaStream_t st) {
    dim3 grid(P.N / P.b, P.BH);
    const size_t smem = bwd_block_smem(P);
#define ELSAA_LAUNCH_BWD(T)                                                    \
    do {                                                                       \
        auto kern = k_bwd_block<T>;                                            \
        cudaFuncSetAttribute(kern,                                             \
                             cudaFuncAttributeMaxDynamicSharedMemorySize,      \
                             (int)smem);                                       \
        kern<<<grid, kBwdThreads, smem, st>>>(                                 \
            (const T *)q, (const T *)k, (const T *)v, (const T *)d_o, w_race,  \
            A, Bm, perm_q, perm_k, lambda_tok, gates, P.N, P.d, P.H, P.b, P.L, \
            P.gamma, P.beta, P.eps, P.scale, P.lambda, P.fusion_mode, dq, dk,  \
            dv, d_gates, d_lambda, gnum, gden, status);                        \
    } while (0)
    if (P.dtype == ELSAA_FP32)
        ELSAA_LAUNCH_BWD(float);
    else
        ELSAA_LAUNCH_BWD(__nv_bfloat16);
#undef ELSAA_LAUNCH_BWD
    return cudaGetLastError();
}

cudaError_t launch_bwd_keys(const Plan &P, const void *k, const void *v,
                            const float *w_race, const float *gA,
                            const float *gB, float *dk, float *dv,
                            cudaStream_t st) {
    dim3 grid((P.N + kKeyTile - 1) / kKeyTile, P.BH);
    const size_t smem = bwd_keys_smem(P);
    if (P.dtype == ELSAA_FP32) {
        auto kern = k_bwd_keys<float>;
        cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             (int)smem);
        kern<<<grid, kKeyThreads, smem, st>>>(
            (const float *)k, (const float *)v, w_race, gA, gB, P.N, P.d, P.H,
            P.L, P.gamma, P.beta, dk, dv);
    } else {
        auto kern = k_bwd_keys<__nv_bfloat16>;
        cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             (int)smem);
        kern<<<grid, kKeyThreads, smem, st>>>(
            (const __nv_bfloat16 *)k, (const __nv_bfloat16 *)v, w_race, gA, gB,
            P.N, P.d, P.H, P.L, P.gamma, P.beta, dk, dv);
    }
    return cudaGetLastError();
}

}  // namespace elsaa
