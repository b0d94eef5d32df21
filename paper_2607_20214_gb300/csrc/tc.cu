// Tensor-core (tcgen05 / TMEM, bf16 in, fp32 accumulate) block attention for
// bf16 inputs whose key blocks span 256 keys (the persistent kernel in
// tc_ws.cu covers b <= 128), plus the support checks of the tensor-core path.
//
//   k_block_attn_tc  one CTA = 128 consecutive sorted query positions:
//                    sortLSH block attention (Algorithm "sortLSH Sparse
//                    Exact Attention Branch", block step), the RACE query
//                    readout (Algorithm RACE, steps 9-10) and the fusion of
//                    Eq. (5)-(6), written at the queries' original rows.
//
// Fusion trick of k_block_attn_tc: the fused row is
//   O_i = c1_i * (P V)_i + c2_i * (Phi_Q B)_i,
//   c1 = g_s m / (l + eps e^-M)      (P = exp(z - M) unnormalised, l = sum P)
//   c2 = g_lr / (L_s (Den + eps)),
// so the features are pre-scaled by c2/c1 and both MMAs accumulate into ONE
// TMEM accumulator; the epilogue multiplies the row by c1.
#include <type_traits>

#include "device_common.cuh"
#include "tc_common.cuh"
#include "tc_race.cuh"

namespace elsaa {

namespace {

using namespace tc;

constexpr int kTcThreads = 256;

// Sparse block attention + RACE readout + fusion for 128 sorted queries.
// 256 threads: thread pairs (tid, tid ^ 128) share a query row (a TMEM lane)
// and split its key columns (softmax), RACE tables (features) and output
// columns (epilogue). NK = keys per query tile (b rounded up to 128).
template <int G, int NK>
__global__ void __launch_bounds__(kTcThreads, NK == 128 ? 2 : 1)
    k_block_attn_tc(const uint16_t *__restrict__ qx,
                    const uint16_t *__restrict__ kx,
                    const uint16_t *__restrict__ vx,
                    const float *__restrict__ w_race,
                    const int32_t *__restrict__ perm_q,
                    const int32_t *__restrict__ perm_k,
                    const float *__restrict__ Ag,
                    const uint16_t *__restrict__ Bh,
                    const float *__restrict__ lambda_tok,
                    const float *__restrict__ gates, uint16_t *__restrict__ ox,
                    float *__restrict__ log_ds_out, float *__restrict__ dlr_out,
                    float *__restrict__ m_out, int N, int d, int H, int b,
                    int L, int Lg_pad, float beta, float eps, float scale,
                    float lambda, int mode, uint32_t tmem_cols,
                    DeviceStatus *status) {
    constexpr int R = 1 << G;
    constexpr int nk = NK;
    extern __shared__ unsigned char smem_raw[];
    __shared__ uint64_t mb;
    __shared__ uint32_t tbase;
    __shared__ int qidx[128];
    __shared__ int kidx[NK];
    __shared__ float xmax[2][128], xsum[2][128], xden[2][128];
    const int p0 = blockIdx.x * 128, bh = blockIdx.y, h = bh % H;
    const int tid = threadIdx.x, warp = tid >> 5;
    const int grp = warp & 3, half = warp >> 2;
    const int row = grp * 32 + (tid & 31);  // query row of the tile
    const int Lg = L * G, r = L * R;
    const int kpos0 = b >= 128 ? (p0 / b) * b : p0;
    const int split = table_split(L, G);
    const int l0 = half ? split : 0, l1 = half ? L : split;

    const uint32_t base = align1k(smem_u32(smem_raw));
    const uint32_t sQ = base;                  // later: B summary [r x d]
    const uint32_t sK = sQ + 128u * d * 2u;
    const uint32_t sV = sK + (uint32_t)nk * d * 2u;  // W first, then V

    if (warp == 0) tmem_alloc(&tbase, tmem_cols);
    if (tid == 0) {
        mbar_init(&mb, 1);
        fence_mbar_init();
    }
    const int32_t *pq = perm_q + (size_t)bh * N;
    const int32_t *pk = perm_k + (size_t)bh * N;
    if (tid < 128) {
        int pos = min(p0 + tid, N - 1);
        int i = pq[pos];
        if (i < 0 || i >= N) {
            report(status, kDevPermRange, 3, bh, i);
            i = 0;
        }
        qidx[tid] = i;
    }
    for (int j = tid; j < nk; j += kTcThreads) {
        int pos = min(kpos0 + j, N - 1);
        int i = pk[pos];
        if (i < 0 || i >= N) {
            report(status, kDevPermRange, 4, bh, i);
            i = 0;
        }
        kidx[j] = i;
    }
    __syncthreads();
    const uint16_t *qh = qx + (size_t)bh * N * d;
    const uint16_t *kh = kx + (size_t)bh * N * d;
    const uint16_t *vh = vx + (size_t)bh * N * d;
    gather_rows(sQ, qh, qidx, 128, d, d, tid, kTcThreads);
    gather_rows(sK, kh, kidx, nk, d, d, tid, kTcThreads);
    cp_async_commit();
    load_planes_bf16(sV, w_race + (size_t)h * Lg * d, Lg, Lg_pad, d, tid,
                     kTcThreads);
    cp_async_wait<0>();
    fence_proxy_async_smem();
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t t = tbase;
    const uint32_t lane = (uint32_t)(grp * 32) << 16;
    const uint32_t colO = (uint32_t)nk;
    if (tid == 0) {
        const uint32_t id_proj = idesc_bf16(128, Lg_pad, false, false);
        const uint32_t id_s = idesc_bf16(128, nk, false, false);
        for (int k = 0; k < d / 16; ++k) {
            uint32_t oq = (k >> 2) * 128 * 128 + (k & 3) * 32;
            uint32_t ow = (k >> 2) * Lg_pad * 128 + (k & 3) * 32;
            uint32_t ok_ = (k >> 2) * nk * 128 + (k & 3) * 32;
            uint64_t aq = smem_desc(sQ + oq, 16, 1024);
            mma_ss(t + colO, aq, smem_desc(sV + ow, 16, 1024), id_proj, k > 0);
            mma_ss(t, aq, smem_desc(sK + ok_, 16, 1024), id_s, k > 0);
        }
        mma_commit(&mb);
    }
    bool ok = mbar_wait(&mb, 0, status, 21);
    ok = __syncthreads_and(ok);  // CTA-uniform from here on
    tc_fence_after();
    // Q, K and W are consumed: stream V into its slot and the bf16 B
    // summary of this head into the Q/K slots while the softmax runs.
    gather_rows(sV, vh, kidx, nk, d, d, tid, kTcThreads);
    load_rows(sQ, Bh + (size_t)bh * r * d, r, d, d, tid, kTcThreads);
    cp_async_commit();

    // ---- RACE features of this row's tables [l0, l1); partial Den
    float sp[32];
    race_bits32(t + lane + colO + l0 * G, (l1 - l0) * G, beta, sp);
    const float *Ah = Ag + (size_t)bh * r;
    float den = 0.0f;
#pragma unroll
    for (int lt = 0; lt < 32 / G; ++lt) {
        if (l0 + lt < l1) {
            float phi[R];
            table_phi<G>(&sp[lt * G], phi);
#pragma unroll
            for (int q = 0; q < R; ++q)
                den = fmaf(phi[q], __ldg(Ah + (l0 + lt) * R + q), den);
        }
    }

    // ---- sparse branch: softmax over this half's key columns
    const float sl2e = scale * kLog2e;
    const int klo = b < 128 ? (row / b) * b : 0;  // the row's key block
    const int khi = b < 128 ? klo + b : nk;
    const int cbeg = half * (nk / 2);
    float mx = -INFINITY;
#pragma unroll
    for (int cc = 0; cc < nk / 2; cc += 32) {
        uint32_t v[32];
        tmem_ld32(t + lane + cbeg + cc, v);
        tmem_wait_ld();
#pragma unroll
        for (int j = 0; j < 32; ++j) {
            const int key = cbeg + cc + j;
            if (key >= klo && key < khi) mx = fmaxf(mx, __uint_as_float(v[j]));
        }
    }
    xmax[half][row] = mx;
    xden[half][row] = den;
    __syncthreads();
    mx = fmaxf(xmax[0][row], xmax[1][row]);
    den = (xden[0][row] + xden[1][row]) * (1.0f / (float)L);
    const float M2 = mx * sl2e;  // row max in log2 units
    float lsum = 0.0f;
    uint32_t ppk[nk / 4];  // this half's P, packed bf16 pairs
#pragma unroll
    for (int cc = 0; cc < nk / 2; cc += 32) {
        uint32_t v[32];
        tmem_ld32(t + lane + cbeg + cc, v);
        tmem_wait_ld();
#pragma unroll
        for (int j = 0; j < 32; j += 2) {
            const int key = cbeg + cc + j;
            float a0 = 0.0f, a1 = 0.0f;
            if (key >= klo && key < khi)
                a0 = ex2_approx(fmaf(__uint_as_float(v[j]), sl2e, -M2));
            if (key + 1 >= klo && key + 1 < khi)
                a1 = ex2_approx(fmaf(__uint_as_float(v[j + 1]), sl2e, -M2));
            lsum += a0 + a1;
            ppk[(cc + j) >> 1] = pack_bf16x2(a0, a1);
        }
    }
    xsum[half][row] = lsum;
    tc_fence_before();
    __syncthreads();  // every S read is done: P may overwrite S
    tc_fence_after();
    lsum = xsum[0][row] + xsum[1][row];
#pragma unroll
    for (int cc = 0; cc < nk / 4; cc += 16)
        tmem_st16(t + lane + (cbeg >> 1) + cc,
                  *reinterpret_cast<uint32_t(*)[16]>(&ppk[cc]));

    // ---- fusion scalars (Eq. (5) in log-sum-exp form, Eq. (6))
    const int qpos = p0 + row;
    const bool qvalid = qpos < N;
    const int qi = qidx[row];
    const size_t tok = (size_t)bh * N + qi;
    const float log_ds = M2 * kLn2 + logf(lsum);
    const float lam = (lambda_tok && qvalid) ? lambda_tok[tok] : lambda;
    const float gs = (gates && qvalid) ? gates[2 * tok] : 1.0f;
    const float gl = (gates && qvalid) ? gates[2 * tok + 1] : 1.0f;
    const float msp = fusion_multiplier(log_ds, lam, den, eps, mode);
    const float c1 = gs * msp / (lsum + eps * ex2_approx(-M2));
    const float c1e = fmaxf(c1, 1e-30f);
    const float c2 = gl / ((float)L * (den + eps));
    const float ratio = c2 / c1e;

    const int r0 = min(r, nk);  // buckets of the first Num pass
    write_phi_tmem<G>(sp, l0, l1, r, ratio, 0, r0, t + lane + (nk >> 1));
    tmem_wait_st();
    cp_async_wait<0>();
    fence_proxy_async_smem();
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    if (tid == 0 && ok) {
        const uint32_t id_o = idesc_bf16(128, d, false, true);
        for (int k = 0; k < nk / 16; ++k)  // O = P V
            mma_ts(t + colO, t + k * 8,
                   smem_desc(sV + k * 2048, (uint32_t)nk * 128, 1024), id_o,
                   k > 0);
        for (int k = 0; k < r0 / 16; ++k)  // O += Phi' B (first buckets)
            mma_ts(t + colO, t + (nk >> 1) + k * 8,
                   smem_desc(sQ + k * 2048, (uint32_t)r * 128, 1024), id_o,
                   1);
        mma_commit(&mb);
    }
    ok = ok && mbar_wait(&mb, 1, status, 22);
    ok = __syncthreads_and(ok);
    tc_fence_after();
    if (r > nk) {  // remaining buckets reuse the P columns
        write_phi_tmem<G>(sp, l0, l1, r, ratio, nk, r, t + lane);
        tmem_wait_st();
        tc_fence_before();
        __syncthreads();
        tc_fence_after();
        if (tid == 0 && ok) {
            const uint32_t id_o = idesc_bf16(128, d, false, true);
            for (int k = 0; k < (r - nk) / 16; ++k)
                mma_ts(t + colO, t + k * 8,
                       smem_desc(sQ + (uint32_t)nk * 128 + k * 2048,
                                 (uint32_t)r * 128, 1024),
                       id_o, 1);
            mma_commit(&mb);
        }
        ok = ok && mbar_wait(&mb, 0, status, 23);  // third completion
        ok = __syncthreads_and(ok);
        tc_fence_after();
    }

    // ---- epilogue: O row = c1 * accumulator, at the original query index
    if (ok) {
        uint16_t *orow = ox + tok * d;
        for (int c = half * (d >> 1); c < (half + 1) * (d >> 1); c += 32) {
            uint32_t v[32];
            tmem_ld32(t + lane + colO + c, v);
            tmem_wait_ld();
            if (qvalid) {
                uint4 *dst = reinterpret_cast<uint4 *>(orow + c);
#pragma unroll
                for (int j = 0; j < 4; ++j) {
                    uint4 w;
                    w.x = pack_bf16x2(c1e * __uint_as_float(v[8 * j]),
                                      c1e * __uint_as_float(v[8 * j + 1]));
                    w.y = pack_bf16x2(c1e * __uint_as_float(v[8 * j + 2]),
                                      c1e * __uint_as_float(v[8 * j + 3]));
                    w.z = pack_bf16x2(c1e * __uint_as_float(v[8 * j + 4]),
                                      c1e * __uint_as_float(v[8 * j + 5]));
                    w.w = pack_bf16x2(c1e * __uint_as_float(v[8 * j + 6]),
                                      c1e * __uint_as_float(v[8 * j + 7]));
                    dst[j] = w;
                }
            }
        }
        if (qvalid && half == 0) {
            if (log_ds_out) log_ds_out[tok] = log_ds;
            if (dlr_out) dlr_out[tok] = den;
            if (m_out) m_out[tok] = msp;
        }
    }
    tc_fence_before();
    __syncthreads();
    if (warp == 0) tmem_dealloc(t, tmem_cols);
}

uint32_t pow2_cols(uint32_t n) {
    uint32_t c = 32;
    while (c < n) c <<= 1;
    return c;
}

template <typename F>
cudaError_t dispatch_gamma(int gamma, F f) {
    switch (gamma) {
        case 1: return f(std::integral_constant<int, 1>());
        case 2: return f(std::integral_constant<int, 2>());
        case 3: return f(std::integral_constant<int, 3>());
        case 4: return f(std::integral_constant<int, 4>());
        case 5: return f(std::integral_constant<int, 5>());
        case 6: return f(std::integral_constant<int, 6>());
        default: return cudaErrorInvalidValue;
    }
}

constexpr int kSmemPerSM = 233472;  // 228 KB of shared memory per SM

// Dynamic shared memory that also caps residency at what TMEM allows.
size_t smem_for(size_t need, uint32_t tmem_cols) {
    int fit = 512 / (int)tmem_cols;  // CTAs whose TMEM fits on one SM
    size_t cap = (size_t)kSmemPerSM / (fit + 1) + 1;
    return need > cap ? need : cap;
}

}  // namespace

bool tc_supported(const Plan &P) {
    if (P.dtype != ELSAA_BF16) return false;
    if (P.d != 64 && P.d != 128) return false;
    if (!(P.b == 32 || P.b == 64 || P.b == 128 || P.b == 256)) return false;
    if (P.gamma > 6 || P.L * P.gamma > 64) return false;
    if (P.r % 16 != 0 || P.r > 256) return false;
    // each half of a row's tables must fit in 32 projection columns
    const int split = table_split(P.L, P.gamma);
    if (split * P.gamma > 32 || (P.L - split) * P.gamma > 32) return false;
    return true;
}

int tc_race_chunks(const Plan &P, int *chunk) {
    // CTAs per SM from the TMEM and shared memory of the key kernel; one
    // wave of chunks over all heads.
    const uint32_t cols = race_keys_ws_cols(P);
    int per_sm = 512 / (int)cols;
    const size_t smem = race_keys_ws_smem(P);
    int by_smem = (int)(kSmemPerSM / (smem + 1024));
    if (by_smem < per_sm) per_sm = by_smem;
    if (per_sm < 1) per_sm = 1;
    long slots = 152L * per_sm;
    int tiles = (P.N + 127) / 128;
    int S = (int)(slots / P.BH);
    if (S < 1) S = 1;
    if (S > tiles) S = tiles;
    int tiles_per = (tiles + S - 1) / S;
    *chunk = tiles_per * 128;
    return (P.N + *chunk - 1) / *chunk;
}

cudaError_t launch_block_attn_tc(
    const Plan &P, const void *q, const void *k, const void *v,
    const float *w_race, const int32_t *perm_q, const int32_t *perm_k,
    const float *A, const uint16_t *Bh, const float *lambda_tok,
    const float *gates, void *o, float *log_d_sparse, float *d_lr,
    float *m_sparse, DeviceStatus *status, cudaStream_t st) {
    const int nk = P.b >= 128 ? P.b : 128;
    const int lg_pad = (P.L * P.gamma + 15) / 16 * 16;
    const uint32_t cols = pow2_cols((uint32_t)(nk + P.d));
    size_t need = 1024 + (size_t)(128 + 2 * nk) * P.d * 2;
    size_t smem = smem_for(need, cols);
    dim3 grid((P.N + 127) / 128, P.BH);
    return dispatch_gamma(P.gamma, [&](auto g) {
        constexpr int G = decltype(g)::value;
        auto run = [&](auto kern) {
            cudaFuncSetAttribute(kern,
                                 cudaFuncAttributeMaxDynamicSharedMemorySize,
                                 (int)smem);
            kern<<<grid, kTcThreads, smem, st>>>(
                (const uint16_t *)q, (const uint16_t *)k, (const uint16_t *)v,
                w_race, perm_q, perm_k, A, Bh, lambda_tok, gates,
                (uint16_t *)o, log_d_sparse, d_lr, m_sparse, P.N, P.d, P.H,
                P.b, P.L, lg_pad, P.beta, P.eps, P.scale, P.lambda,
                P.fusion_mode, cols, status);
            return cudaGetLastError();
        };
        return nk == 256 ? run(k_block_attn_tc<G, 256>)
                         : run(k_block_attn_tc<G, 128>);
    });
}

}  // namespace elsaa
