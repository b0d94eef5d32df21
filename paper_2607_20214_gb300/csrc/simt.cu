// CUDA-core (fp32) kernels of the RACE branch, the sortLSH block attention
// and the fusion epilogue. These serve fp32 inputs (where tensor-core
// rounding would exceed an fp32 tolerance) and every dtype when
// params.impl == ELSAA_IMPL_SIMT.
#include "device_common.cuh"

namespace elsaa {

namespace {

// ---------------------------------------------------------------------------
// RACE key side (Algorithm "RACE Low-Rank Attention Branch", steps 3-7):
// partial bucket summaries A^(l) = Phi_K^T 1 and B^(l) = Phi_K^T V over one
// chunk of keys, for one slice of at most 64 buckets (whole tables).
// Grid (S chunks, slices, BH heads); output part[bh][s] = [r x d] B then [r] A.
// The same kernel forms the backward pass's gB = sum_i phi(Q_i) gNum_i^T and
// gA = sum_i phi(Q_i) gDen_i: values of type TV (fp32 there) and an optional
// per-token weight wA of the A sum (NULL: 1).
constexpr int kRaceThreads = 256;
constexpr int kRaceTok = 32;  // keys staged per iteration

template <typename T, typename TV>
__global__ void __launch_bounds__(kRaceThreads)
    k_race_partial(const T *__restrict__ kx, const TV *__restrict__ vx,
                   const float *__restrict__ wA,
                   const float *__restrict__ w_race, int N, int d, int H,
                   int L, int gamma, int tps, int chunk, float beta,
                   float *__restrict__ part) {
    extern __shared__ float smem[];
    const int s = blockIdx.x, slice = blockIdx.y, bh = blockIdx.z;
    const int S = gridDim.x;
    const int tid = threadIdx.x;
    const int h = bh % H;
    const int R = 1 << gamma;
    const int r = L * R;
    const int t0 = slice * tps;
    const int t1 = min(L, t0 + tps);
    const int nb = (t1 - t0) * R;  // buckets in this slice (<= 64)
    const int ds = d + 1;
    float *kt = smem;                  // [kRaceTok][d + 1]
    float *vt = kt + kRaceTok * ds;    // [kRaceTok][d]
    float *ph = vt + kRaceTok * d;     // [kRaceTok][64]
    float *wr = ph + kRaceTok * 64;    // [tables in slice][gamma][d]
    __shared__ float wt[kRaceTok];     // A weights of the staged tokens

    for (int i = tid; i < (t1 - t0) * gamma * d; i += kRaceThreads)
        wr[i] = w_race[((size_t)h * L + t0) * gamma * d + i];

    // accumulator ownership: dim e = tid % d, buckets rb = grp + j * ngrp
    const int ngrp = kRaceThreads / d;
    const int e = tid % d, grp = tid / d;
    const int nacc = (nb + ngrp - 1) / ngrp;  // <= 64 / (256 / d) <= 32
    float acc[32];
#pragma unroll
    for (int j = 0; j < 32; ++j) acc[j] = 0.f;
    float accA = 0.f;

    const T *kh = kx + (size_t)bh * N * d;
    const TV *vh = vx + (size_t)bh * N * d;
    const int c0 = s * chunk;
    const int c1 = min(N, c0 + chunk);
    for (int base = c0; base < c1; base += kRaceTok) {
        __syncthreads();
        for (int i = tid; i < kRaceTok * d; i += kRaceThreads) {
            int row = i / d, col = i - row * d;
            int n = base + row;
            bool ok = n < c1;
            kt[row * ds + col] = ok ? to_f32<T>(kh[(size_t)n * d + col]) : 0.f;
            vt[row * d + col] = ok ? to_f32<TV>(vh[(size_t)n * d + col]) : 0.f;
        }
        if (tid < kRaceTok) {
            const int n = base + tid;
            wt[tid] = n < c1 ? (wA ? wA[(size_t)bh * N + n] : 1.f) : 0.f;
        }
        __syncthreads();
        // features: one task per (token, table)
        for (int task = tid; task < kRaceTok * (t1 - t0); task += kRaceThreads) {
            int tok = task % kRaceTok, tl = task / kRaceTok;
            float *out = ph + tok * 64 + tl * R;
            if (base + tok >= c1) {
                for (int rr = 0; rr < R; ++rr) out[rr] = 0.f;
                continue;
            }
            float sp[8], sn[8];
            const float *xr = kt + tok * ds;
            for (int bb = 0; bb < gamma; ++bb) {
                const float *w = wr + (tl * gamma + bb) * d;
                float a = 0.f;
                for (int i = 0; i < d; ++i) a = fmaf(w[i], xr[i], a);
                race_bit_factors(a, beta, sp[bb], sn[bb]);
            }
            for (int rr = 0; rr < R; ++rr) {
                float pr = 1.f;
                for (int bb = 0; bb < gamma; ++bb)
                    pr *= ((rr >> bb) & 1) ? sp[bb] : sn[bb];
                out[rr] = pr;
            }
        }
        __syncthreads();
        for (int tok = 0; tok < kRaceTok; ++tok) {
            float vv = vt[tok * d + e];
            const float *pr = ph + tok * 64;
#pragma unroll
            for (int j = 0; j < 32; ++j) {
                int rb = grp + j * ngrp;
                if (j < nacc && rb < nb) acc[j] = fmaf(pr[rb], vv, acc[j]);
            }
            if (tid < nb) accA = fmaf(pr[tid], wt[tok], accA);
        }
    }
    float *out = part + ((size_t)bh * S + s) * ((size_t)r * d + r);
#pragma unroll
    for (int j = 0; j < 32; ++j) {
        int rb = grp + j * ngrp;
        if (j < nacc && rb < nb) out[(size_t)(t0 * R + rb) * d + e] = acc[j];
    }
    if (tid < nb) out[(size_t)r * d + t0 * R + tid] = accA;
}

// Fixed-order (deterministic) sum of the S chunk partials.
__global__ void k_race_reduce(const float *__restrict__ part, int S, int r,
                              int d, float *__restrict__ A,
                              float *__restrict__ Bm, uint16_t *__restrict__ Bh) {
    const int bh = blockIdx.y;
    const size_t per = (size_t)r * d + r;
    for (size_t i = (size_t)blockIdx.x * blockDim.x + threadIdx.x; i < per;
         i += (size_t)gridDim.x * blockDim.x) {
        const float *p = part + (size_t)bh * S * per + i;
        float s = 0.f;
        for (int c = 0; c < S; ++c) s += p[(size_t)c * per];
        if (i < (size_t)r * d) {
            Bm[(size_t)bh * r * d + i] = s;
            if (Bh) {
                __nv_bfloat16 hb = __float2bfloat16_rn(s);
                Bh[(size_t)bh * r * d + i] = *reinterpret_cast<uint16_t *>(&hb);
            }
        } else {
            A[(size_t)bh * r + (i - (size_t)r * d)] = s;
        }
    }
}

// ---------------------------------------------------------------------------
// sortLSH block attention + RACE query readout + fusion, CUDA cores, fp32.
// One CTA = 32 consecutive sorted query positions (inside one block, since
// b % 32 == 0). Per query: online-softmax pass over the b keys of its key
// block (Algorithm sortLSH, block step) -> O_sparse, log d_sparse; features
// phi(Q_i) and Num/Den from the summaries (Algorithm RACE, steps 9-10);
// Eq. (5)-(6) fusion; row written at the query's original index (un-permute).
constexpr int kBlkThreads = 256;
constexpr int kQPerWarp = kSimtQT / (kBlkThreads / 32);  // 4
constexpr int kKC = 32;  // keys per staged chunk

template <typename T>
__global__ void __launch_bounds__(kBlkThreads)
    k_block_attn(const T *__restrict__ qx, const T *__restrict__ kx,
                 const T *__restrict__ vx, const float *__restrict__ w_race,
                 const int32_t *__restrict__ perm_q,
                 const int32_t *__restrict__ perm_k,
                 const float *__restrict__ Ag, const float *__restrict__ Bg,
                 const float *__restrict__ lambda_tok,
                 const float *__restrict__ gates, T *__restrict__ ox,
                 float *__restrict__ o32,
                 float *__restrict__ log_ds_out, float *__restrict__ dlr_out,
                 float *__restrict__ m_out, int N, int d, int H, int b,
                 int L, int gamma, int tps, int nb, float beta, float eps,
                 float scale, float lambda, int mode, DeviceStatus *status,
                 const int32_t *__restrict__ cand,
                 const uint32_t *__restrict__ selmask, int tk_c) {
    extern __shared__ float smem[];
    const int bh = blockIdx.y, h = bh % H;
    const int pos0 = blockIdx.x * kSimtQT;
    const int blk = pos0 / b;
    const int tid = threadIdx.x, lane = tid & 31, wid = tid >> 5;
    const int R = 1 << gamma, r = L * R;
    const int ds = d + 1;
    float *qs = smem;                 // [32][d]
    float *ks = qs + kSimtQT * d;     // [32][d + 1]
    float *vs = ks + kKC * ds;        // [32][d]
    __shared__ int qidx[kSimtQT];
    __shared__ float s_logds[kSimtQT], s_den[kSimtQT], s_m[kSimtQT];

    const T *qh = qx + (size_t)bh * N * d;
    const T *kh = kx + (size_t)bh * N * d;
    const T *vh = vx + (size_t)bh * N * d;
    const int32_t *pq = perm_q + (size_t)bh * N;
    const int32_t *pk = perm_k + (size_t)bh * N;

    if (tid < kSimtQT) {
        int i = pq[pos0 + tid];
        if (i < 0 || i >= N) {
            report(status, kDevPermRange, 1, bh, i);
            i = 0;
        }
        qidx[tid] = i;
    }
    __syncthreads();
    for (int i = tid; i < kSimtQT * d; i += kBlkThreads) {
        int row = i / d, col = i - row * d;
        qs[i] = to_f32<T>(qh[(size_t)qidx[row] * d + col]);
    }

    // ---- sparse branch: online softmax over the key block
    const int nd = d / 32;  // dims per lane (1, 2 or 4)
    float m_run[kQPerWarp], l_run[kQPerWarp], o_acc[kQPerWarp][4];
#pragma unroll
    for (int qq = 0; qq < kQPerWarp; ++qq) {
        m_run[qq] = -INFINITY;
        l_run[qq] = 0.f;
#pragma unroll
        for (int c = 0; c < 4; ++c) o_acc[qq][c] = 0.f;
    }
    // key block blk and its nb neighbouring sorted blocks on each side,
    // clipped to the N / b blocks: sorted positions [lo b, (hi + 1) b).
    // With the top-k selector: the tk_c candidate blocks of the query
    // block, each key masked unless the query selected it.
    const int nblk = N / b;
    const int lo = blk - nb > 0 ? blk - nb : 0;
    const int hi = blk + nb < nblk - 1 ? blk + nb : nblk - 1;
    const int kbase = lo * b;
    const int nkeys = cand ? tk_c * b : (hi - lo + 1) * b;
    const int32_t *cb = cand ? cand + ((size_t)bh * nblk + blk) * tk_c
                             : nullptr;
    const int W = tk_c * b / 32;  // mask words per query (selector 1)
    for (int c0 = 0; c0 < nkeys; c0 += kKC) {
        __syncthreads();
        // sorted key position of chunk c0 (chunks never straddle a block:
        // b is a multiple of kKC)
        int kp0 = kbase + c0;
        if (cb) {
            int u = cb[c0 / b];
            if (u < 0 || u >= nblk) {
                report(status, kDevPermRange, 3, bh, u);
                u = blk;
            }
            kp0 = u * b + c0 % b;
        }
        for (int i = tid; i < kKC * d; i += kBlkThreads) {
            int row = i / d, col = i - row * d;
            int j = pk[kp0 + row];
            if (j < 0 || j >= N) {
                if (col == 0) report(status, kDevPermRange, 2, bh, j);
                j = 0;
            }
            ks[row * ds + col] = to_f32<T>(kh[(size_t)j * d + col]);
            vs[row * d + col] = to_f32<T>(vh[(size_t)j * d + col]);
        }
        __syncthreads();
#pragma unroll
        for (int qq = 0; qq < kQPerWarp; ++qq) {
            const float *qr = qs + (wid * kQPerWarp + qq) * d;
            const float *kr = ks + lane * ds;
            float z = 0.f;
            for (int e = 0; e < d; ++e) z = fmaf(qr[e], kr[e], z);
            z *= scale;
            bool keep = true;
            if (selmask)
                keep = (selmask[((size_t)bh * N + pos0 + wid * kQPerWarp +
                                 qq) * W + c0 / 32] >> lane) & 1u;
            if (!keep) z = -INFINITY;
            float mnew = fmaxf(m_run[qq], warp_max(z));
            // nothing kept yet (mnew = -inf): no change
            float alpha = mnew == -INFINITY ? 1.0f : expf(m_run[qq] - mnew);
            float p = keep ? expf(z - mnew) : 0.0f;
            l_run[qq] = l_run[qq] * alpha + warp_sum(p);
#pragma unroll
            for (int c = 0; c < 4; ++c) o_acc[qq][c] *= alpha;
            for (int j = 0; j < kKC; ++j) {
                float pj = __shfl_sync(0xffffffffu, p, j);
#pragma unroll
                for (int c = 0; c < 4; ++c)
                    if (c < nd)
                        o_acc[qq][c] = fmaf(pj, vs[j * d + lane + 32 * c],
                                            o_acc[qq][c]);
            }
            m_run[qq] = mnew;
        }
    }
    __syncthreads();
    // O_sparse = sum exp(z) v / (d_s + eps), d_s = exp(m) l.
    float *os = ks;  // [32][d] reuse: sparse outputs
#pragma unroll
    for (int qq = 0; qq < kQPerWarp; ++qq) {
        const int row = wid * kQPerWarp + qq;
        float inv = 1.0f / (l_run[qq] + eps * expf(-m_run[qq]));
#pragma unroll
        for (int c = 0; c < 4; ++c)
            if (c < nd) os[row * d + lane + 32 * c] = o_acc[qq][c] * inv;
        if (lane == 0) s_logds[row] = m_run[qq] + logf(l_run[qq]);
    }

    // ---- RACE readout for the 32 queries, slice by slice of tables
    float *phq = vs;                   // [32][64] features of the slice
    float *wr = phq + kSimtQT * 64;    // [tps][gamma][d]
    const int ngrp = kBlkThreads / d;
    const int e = tid % d, grp = tid / d;
    const int nq = kSimtQT / ngrp;     // queries per thread (<= 32)
    float num[32];
#pragma unroll
    for (int j = 0; j < 32; ++j) num[j] = 0.f;
    float den = 0.f;
    const float *Ah = Ag + (size_t)bh * r;
    const float *Bh = Bg + (size_t)bh * r * d;
    for (int t0 = 0; t0 < L; t0 += tps) {
        const int t1 = min(L, t0 + tps);
        const int nb = (t1 - t0) * R;
        __syncthreads();
        for (int i = tid; i < (t1 - t0) * gamma * d; i += kBlkThreads)
            wr[i] = w_race[((size_t)h * L + t0) * gamma * d + i];
        __syncthreads();
        for (int task = tid; task < kSimtQT * (t1 - t0); task += kBlkThreads) {
            int qrow = task % kSimtQT, tl = task / kSimtQT;
            const float *xr = qs + qrow * d;
            float sp[8], sn[8];
            for (int bb = 0; bb < gamma; ++bb) {
                const float *w = wr + (tl * gamma + bb) * d;
                float a = 0.f;
                for (int i = 0; i < d; ++i) a = fmaf(w[i], xr[i], a);
                race_bit_factors(a, beta, sp[bb], sn[bb]);
            }
            for (int rr = 0; rr < R; ++rr) {
                float pr = 1.f;
                for (int bb = 0; bb < gamma; ++bb)
                    pr *= ((rr >> bb) & 1) ? sp[bb] : sn[bb];
                phq[qrow * 64 + tl * R + rr] = pr;
            }
        }
        __syncthreads();
        for (int rb = 0; rb < nb; ++rb) {
            float bv = Bh[(size_t)(t0 * R + rb) * d + e];
#pragma unroll
            for (int j = 0; j < 32; ++j)
                if (j < nq) num[j] = fmaf(phq[(grp + j * ngrp) * 64 + rb], bv,
                                         num[j]);
        }
        if (tid < kSimtQT)
            for (int rb = 0; rb < nb; ++rb)
                den = fmaf(phq[tid * 64 + rb], Ah[t0 * R + rb], den);
    }
    const float invL = 1.0f / (float)L;
    if (tid < kSimtQT) {
        const int i = qidx[tid];
        const size_t tok = (size_t)bh * N + i;
        float dl = den * invL;
        float lam = lambda_tok ? lambda_tok[tok] : lambda;
        float mm = fusion_multiplier(s_logds[tid], lam, dl, eps, mode);
        s_den[tid] = dl;
        s_m[tid] = mm;
        if (log_ds_out) log_ds_out[tok] = s_logds[tid];
        if (dlr_out) dlr_out[tok] = dl;
        if (m_out) m_out[tok] = mm;
    }
    __syncthreads();
#pragma unroll
    for (int j = 0; j < 32; ++j) {
        if (j >= nq) break;
        const int row = grp + j * ngrp;
        const int i = qidx[row];
        const size_t tok = (size_t)bh * N + i;
        float gs = gates ? gates[tok * 2] : 1.f;
        float gl = gates ? gates[tok * 2 + 1] : 1.f;
        float olr = (num[j] * invL) / (s_den[row] + eps);
        float val = gs * s_m[row] * os[row * d + e] + gl * olr;
        if (o32)
            o32[tok * d + e] = val;
        else
            ox[tok * d + e] = from_f32<T>(val);
    }
}

}  // namespace

cudaError_t launch_race_partial_simt(const Plan &P, const void *k,
                                     const void *v, const float *w_race,
                                     float *part, cudaStream_t st) {
    dim3 grid(P.S, P.slices, P.BH);
    size_t smem = sizeof(float) *
                  ((size_t)kRaceTok * (P.d + 1) + (size_t)kRaceTok * P.d +
                   (size_t)kRaceTok * 64 +
                   (size_t)P.tables_per_slice * P.gamma * P.d);
    if (P.dtype == ELSAA_FP32) {
        auto kern = k_race_partial<float, float>;
        cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             (int)smem);
        kern<<<grid, kRaceThreads, smem, st>>>(
            (const float *)k, (const float *)v, nullptr, w_race, P.N, P.d,
            P.H, P.L, P.gamma, P.tables_per_slice, P.chunk, P.beta, part);
    } else {
        auto kern = k_race_partial<__nv_bfloat16, __nv_bfloat16>;
        cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             (int)smem);
        kern<<<grid, kRaceThreads, smem, st>>>(
            (const __nv_bfloat16 *)k, (const __nv_bfloat16 *)v, nullptr,
            w_race, P.N, P.d, P.H, P.L, P.gamma, P.tables_per_slice, P.chunk,
            P.beta, part);
    }
    return cudaGetLastError();
}

cudaError_t launch_race_partial_weighted(const Plan &P, const void *x,
                                         const float *vals, const float *wA,
                                         const float *w_race, float *part,
                                         cudaStream_t st) {
    dim3 grid(P.S, P.slices, P.BH);
    size_t smem = sizeof(float) *
                  ((size_t)kRaceTok * (P.d + 1) + (size_t)kRaceTok * P.d +
                   (size_t)kRaceTok * 64 +
                   (size_t)P.tables_per_slice * P.gamma * P.d);
    if (P.dtype == ELSAA_FP32) {
        auto kern = k_race_partial<float, float>;
        cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             (int)smem);
        kern<<<grid, kRaceThreads, smem, st>>>(
            (const float *)x, vals, wA, w_race, P.N, P.d, P.H, P.L, P.gamma,
            P.tables_per_slice, P.chunk, P.beta, part);
    } else {
        auto kern = k_race_partial<__nv_bfloat16, float>;
        cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             (int)smem);
        kern<<<grid, kRaceThreads, smem, st>>>(
            (const __nv_bfloat16 *)x, vals, wA, w_race, P.N, P.d, P.H, P.L,
            P.gamma, P.tables_per_slice, P.chunk, P.beta, part);
    }
    return cudaGetLastError();
}

// k_race_reduce four values per thread (per and r d multiples of 4): the
// same sums in the same chunk order, 16-byte loads and stores.
__global__ void k_race_reduce4(const float *__restrict__ part, int S, int r,
                               int d, float *__restrict__ A,
                               float *__restrict__ Bm,
                               uint16_t *__restrict__ Bh) {
    const int bh = blockIdx.y;
    const size_t per = (size_t)r * d + r, rd = (size_t)r * d;
    for (size_t i = 4 * ((size_t)blockIdx.x * blockDim.x + threadIdx.x);
         i < per; i += 4 * (size_t)gridDim.x * blockDim.x) {
        const float *p = part + (size_t)bh * S * per + i;
        float4 s = make_float4(0.f, 0.f, 0.f, 0.f);
        for (int c = 0; c < S; ++c) {
            const float4 x =
                *reinterpret_cast<const float4 *>(p + (size_t)c * per);
            s.x += x.x;
            s.y += x.y;
            s.z += x.z;
            s.w += x.w;
        }
        if (i < rd) {
            *reinterpret_cast<float4 *>(Bm + (size_t)bh * rd + i) = s;
            if (Bh) {
                const __nv_bfloat162 lo = __floats2bfloat162_rn(s.x, s.y);
                const __nv_bfloat162 hi = __floats2bfloat162_rn(s.z, s.w);
                uint2 w;
                w.x = *reinterpret_cast<const uint32_t *>(&lo);
                w.y = *reinterpret_cast<const uint32_t *>(&hi);
                *reinterpret_cast<uint2 *>(Bh + (size_t)bh * rd + i) = w;
            }
        } else {
            *reinterpret_cast<float4 *>(A + (size_t)bh * r + (i - rd)) = s;
        }
    }
}

cudaError_t launch_race_reduce(const Plan &P, const float *part, float *A,
                               float *Bm, uint16_t *Bh, cudaStream_t st) {
    size_t per = (size_t)P.r * P.d + P.r;
    if (per % 4 == 0 && ((size_t)P.r * P.d) % 4 == 0 && P.r % 4 == 0) {
        int gx = (int)((per / 4 + 255) / 256);
        if (gx > 1024) gx = 1024;
        k_race_reduce4<<<dim3(gx, P.BH), 256, 0, st>>>(part, P.S, P.r, P.d,
                                                        A, Bm, Bh);
        return cudaGetLastError();
    }
    int gx = (int)((per + 255) / 256);
    if (gx > 1024) gx = 1024;
    dim3 grid(gx, P.BH);
    k_race_reduce<<<grid, 256, 0, st>>>(part, P.S, P.r, P.d, A, Bm, Bh);
    return cudaGetLastError();
}

cudaError_t launch_block_attn_simt(
    const Plan &P, const void *q, const void *k, const void *v,
    const float *w_race, const int32_t *perm_q, const int32_t *perm_k,
    const float *A, const float *Bm, const float *lambda_tok,
    const float *gates, void *o, float *log_d_sparse, float *d_lr,
    float *m_sparse, DeviceStatus *status, cudaStream_t st,
    const int32_t *cand, const uint32_t *selmask) {
    dim3 grid(P.N / kSimtQT, P.BH);
    // phase 1: qs + ks(padded) + vs; phase 2 reuses ks, vs for outputs,
    // features and planes.
    size_t ph1 = (size_t)kSimtQT * P.d + (size_t)kKC * (P.d + 1) +
                 (size_t)kKC * P.d;
    size_t ph2 = (size_t)kSimtQT * P.d + (size_t)kKC * (P.d + 1) +
                 (size_t)kSimtQT * 64 +
                 (size_t)P.tables_per_slice * P.gamma * P.d;
    size_t smem = sizeof(float) * (ph1 > ph2 ? ph1 : ph2);
#define ELSAA_LAUNCH_BLK(T)                                                   \
    do {                                                                      \
        auto kern = k_block_attn<T>;                                          \
        cudaFuncSetAttribute(kern,                                            \
                             cudaFuncAttributeMaxDynamicSharedMemorySize,     \
                             (int)smem);                                      \
        kern<<<grid, kBlkThreads, smem, st>>>(                                \
            (const T *)q, (const T *)k, (const T *)v, w_race, perm_q, perm_k, \
            A, Bm, lambda_tok, gates, P.o32 ? nullptr : (T *)o,               \
            P.o32 ? (float *)o : nullptr, log_d_sparse, d_lr, m_sparse,       \
            P.N, P.d, P.H, P.b, P.L, P.gamma, P.tables_per_slice, P.nb,       \
            P.beta, P.eps, P.scale, P.lambda, P.fusion_mode, status, cand,    \
            selmask, P.tk_c);                                                 \
    } while (0)
    if (P.dtype == ELSAA_FP32)
        ELSAA_LAUNCH_BLK(float);
    else
        ELSAA_LAUNCH_BLK(__nv_bfloat16);
#undef ELSAA_LAUNCH_BLK
    return cudaGetLastError();
}

}  // namespace elsaa
