// Tensor-core backward of the sparse branch and of the RACE query side
// (bf16 inputs, b = 64, d_h = 64, gamma = 4, L_s in {4, 8}): the derivative
// of Algorithm "sortLSH Sparse Exact Attention Branch" (block step), of the
// RACE readout (Algorithm "RACE Low-Rank Attention Branch", steps 9-10) and
// of the fusion, Eq. (5)-(6), the same quantities as k_bwd_block.
//
// One persistent CTA per SM walks 128-query tiles (two sorted blocks of 64)
// ordered by head. Per tile, with operands in shared memory (bf16, 128-byte
// swizzled panels; transposes are MN-major views of the same bytes) and
// accumulators in tensor memory:
//   MMA  [Z | U]  = Q [K ; W]^T          scores and RACE projections
//   CUDA E = exp(scale Z - M) on each query's own block (the other block's
//        keys are zero), l, features phi(Q) and Den
//   MMA  Y = E V,  Num = phi B
//   CUDA per-query scalars (Eq. (5)-(6) backward), X = gN_s e^M = c_x G,
//        gNum = G g_lr / (Den + eps)
//   MMA  dV = E^T X,  P = X V^T,  Gphi = gNum B^T,
//        [gB | gA] += phi^T [gNum | dL/dDen]  (summed over the CTA's tiles
//        of one head in tensor memory)
//   CUDA dZ = scale E (P + e^M dL/dd_s), dL/dphi = (Gphi + A dL/dDen) / L,
//        back through the corner softmax and tanh -> dL/d(W q)
//   MMA  dQ = dZ K + dL/d(W q) W,  dK = dZ^T Q
// Every key belongs to exactly one block, so dV, dK (sparse part) are
// plain stores; the RACE key side adds to them afterwards. The per-head
// sums gB, gA that the key side needs leave the kernel as one partial per
// (head, CTA that worked on the head); the key-side kernel sums them in a
// fixed order when it starts on the head.
// Operands in bf16 (relative rounding 2^-9), accumulation in fp32.
#include "device_common.cuh"
#include "tc_common.cuh"
#include "tc_race.cuh"

namespace elsaa {

namespace {

using namespace tc;

constexpr int kBtThreads = 256;
constexpr int kBtT = 128;  // queries (and keys) of a tile: two blocks of 64
constexpr int kBtD = 64;   // d_h
// persistent CTAs of the block kernel: one per SM of a GB300 (fixed, so the
// workspace size does not depend on the device the plan is made on)
constexpr int kBtGrid = 152;
// TMEM columns (512 allocated)
constexpr uint32_t kCS = 0;      // scores [0, 128), projections [128, 160)
constexpr uint32_t kCO = 160;    // E V, then dQ
constexpr uint32_t kCN = 224;    // phi B, then dK
constexpr uint32_t kCG = 160;    // gNum B^T (r <= 128 columns) between them
constexpr uint32_t kCdV = 288;   // E^T X
constexpr uint32_t kCAcc = 352;  // [gB | gA] of the current head, d + 16

// The 16 entries of one table's summary (a 64-byte aligned run in shared
// memory) in four 16-byte loads.
__device__ __forceinline__ void load_table16(const float *a, float (&x)[16]) {
    const float4 *p = reinterpret_cast<const float4 *>(a);
#pragma unroll
    for (int q = 0; q < 4; ++q) {
        const float4 w = p[q];
        x[4 * q] = w.x;
        x[4 * q + 1] = w.y;
        x[4 * q + 2] = w.z;
        x[4 * q + 3] = w.w;
    }
}

__device__ __forceinline__ void unpack_bf16x8(const uint4 &u, float *x) {
    const uint32_t w[4] = {u.x, u.y, u.z, u.w};
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        x[2 * i] = __uint_as_float(w[i] << 16);
        x[2 * i + 1] = __uint_as_float(w[i] & 0xffff0000u);
    }
}

// Per-bit factors of a table with the tanh approximation (as the forward's
// tensor-core kernels): sp = sigma(2 beta tanh u) = 1/2 + tanh(beta tanh u)/2,
// sn = 1 - sp; tu = tanh u (for the derivative of the projection).
__device__ __forceinline__ void bit_factors_fast(float u, float beta,
                                                 float &sp, float &sn,
                                                 float &tu) {
    tu = tanh_approx(u);
    const float t = tanh_approx(beta * tu);
    sp = fmaf(0.5f, t, 0.5f);
    sn = fmaf(-0.5f, t, 0.5f);
}

__device__ __forceinline__ float lse2f(float a, float b) {
    const float mx = fmaxf(a, b);
    if (mx == -INFINITY) return -INFINITY;
    return mx + __logf(__expf(a - mx) + __expf(b - mx));
}

template <int L>
__global__ void __launch_bounds__(kBtThreads, 1)
    k_bwd_block_tc(const uint16_t *__restrict__ qx,
                   const uint16_t *__restrict__ kx,
                   const uint16_t *__restrict__ vx,
                   const uint16_t *__restrict__ gx,
                   const uint16_t *__restrict__ w_bf16,
                   const uint16_t *__restrict__ Bh,
                   const float *__restrict__ Ag,
                   const int32_t *__restrict__ perm_q,
                   const int32_t *__restrict__ perm_k,
                   const float *__restrict__ lambda_tok,
                   const float *__restrict__ gates, int N, int H,
                   float beta, float eps, float scale, float lambda, int mode,
                   int tiles_per_head, long total_tiles,
                   float *__restrict__ dq, float *__restrict__ dk,
                   float *__restrict__ dv, float *__restrict__ d_gates,
                   float *__restrict__ d_lambda, float *__restrict__ part,
                   int S_seg, DeviceStatus *status) {
    constexpr int R = 16, G = 4;
    constexpr int r = L * R, Lg = L * G;
    constexpr int Lg_pad = (Lg + 15) / 16 * 16;
    constexpr int NR = kBtT + Lg_pad;  // key rows + plane rows
    constexpr int TL = L / 2;          // tables per row half
    constexpr int d = kBtD;
    extern __shared__ unsigned char smem_raw[];
    __shared__ uint64_t mma_bar, sums_bar;
    __shared__ uint32_t tbase;
    __shared__ int abort_flag;
    __shared__ float xa[2][kBtT], xb[2][kBtT], xc[2][kBtT];
    __shared__ int qrow2[2][kBtT], krow2[2][kBtT];  // by tile parity
    volatile int *abort = &abort_flag;
    const int tid = threadIdx.x, warp = tid >> 5, lane_id = tid & 31;
    const int half = warp >> 2;
    const int row = (warp & 3) * 32 + lane_id;  // TMEM lane
    const uint32_t lane = (uint32_t)((warp & 3) * 32) << 16;

    const uint32_t base = align1k(smem_u32(smem_raw));
    // Q [128 x 64] and [K ; W] [NR x 64] of two tiles, by tile parity: the
    // next tile's rows land while this one computes
    const uint32_t kQKW = 16384 + align1k(NR * 128);
    // [128 x r]; the bucket-sum MMA reads 128 bucket columns, so with
    // r = 64 its unused upper half reads the 16 KB after sPhi (sG)
    const uint32_t sPhi = base + 2 * kQKW;
    const uint32_t sG = sPhi + align1k(kBtT * r * 2);  // dO, then X = c_x dO
    const uint32_t sGN = sG + 16384;                // [128 x 64]
    const uint32_t sDU = sGN + 16384;  // dL/dDen (columns 0-15), dL/du (32-63)
    const uint32_t sV = sDU + 16384;                // [128 x 64]
    const uint32_t sE = sV + 16384;                 // [128 x 128]: E, dZ
    const uint32_t sB = sE + 32768;                 // [r x 64]
    const uint32_t sAo = sB + align1k(r * 128);     // fp32 [r]
    const float *Asm =
        reinterpret_cast<const float *>(smem_raw + (sAo - smem_u32(smem_raw)));

    const long t_begin = total_tiles * blockIdx.x / gridDim.x;
    const long t_end = total_tiles * (blockIdx.x + 1) / gridDim.x;

    if (warp == 0) tmem_alloc(&tbase, 512);
    if (tid == 0) {
        mbar_init(&mma_bar, 1);
        mbar_init(&sums_bar, 1);
        abort_flag = 0;
        fence_mbar_init();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tm = tbase;
    uint32_t mph = 0, sph = 0;  // barrier phases completed
    // everyone waits for a commit of thread 0
    auto mma_wait = [&](uint64_t *bar, uint32_t &ph, int site) -> bool {
        const bool ok = mbar_wait_or_abort(bar, ph & 1, abort, status, site);
        ++ph;
        tc_fence_after();
        return __syncthreads_and(ok);
    };
    // thread 0 issues, everyone waits for the commit
    auto mma_done = [&](int site) -> bool {
        if (tid == 0) mma_commit(&mma_bar);
        return mma_wait(&mma_bar, mph, site);
    };
    // 16-byte chunk (8 bf16) at (row, chunk) of a panel region of `rows`
    auto st8 = [&](uint32_t region, int rr, int chunk, int rows,
                   const float *v) {
        st_shared_bf16x8(region + panel_offset(rr, chunk, rows), v);
    };
    auto ld8 = [&](uint32_t region, int rr, int chunk, int rows, float *v) {
        unpack_bf16x8(ld_shared_v4(region + panel_offset(rr, chunk, rows)),
                      v);
    };
    // fp32 gradient rows leave through shared memory: each thread stages
    // its 32 TMEM columns into its row (256 bytes, the 16-byte chunks
    // XOR-permuted by row & 7 so that eight consecutive rows hit eight
    // bank groups), then every warp writes whole rows, two per
    // instruction, to their original positions.
    static_assert(kBtD == 64, "staged rows are 256 bytes");
    auto stage_f32 = [&](uint32_t region, const uint32_t *v) {
        const uint32_t rb = region + (uint32_t)row * 256;
#pragma unroll
        for (int q = 0; q < 8; ++q)
            st_shared_v4(rb + ((uint32_t)((8 * half + q) ^ (row & 7)) << 4),
                         v[4 * q], v[4 * q + 1], v[4 * q + 2], v[4 * q + 3]);
    };
    auto flush_f32 = [&](uint32_t region, float *dst, const int *rows) {
        const int c = lane_id & 15;
#pragma unroll
        for (int it = 0; it < kBtT / (2 * kBtThreads / 32); ++it) {
            const int i = (2 * kBtThreads / 32) * it + 2 * warp + (lane_id >> 4);
            const uint4 w =
                ld_shared_v4(region + (uint32_t)i * 256 +
                             ((uint32_t)(c ^ (i & 7)) << 4));
            *reinterpret_cast<uint4 *>(dst + (size_t)rows[i] * d + 4 * c) = w;
        }
    };

    // Rows of tile tt (sorted positions -> original rows) into the index
    // arrays of parity tt & 1, from permutation entries fetched into
    // registers a tile earlier. The next tile's copies start as soon as
    // their buffers are free: Q and K (other parity) in phase 1, V after
    // phase 5, the head's B and A and then dO in phase 7. The top of a tile
    // waits for all but the newest copy group (dO), phase 4 for dO.
    int qi_next = 0, ki_next = 0;
    auto fetch_rows = [&](long tt) {
        if (tid < kBtT) {
            const int bh = (int)(tt / tiles_per_head);
            const size_t p = (size_t)bh * N +
                             (size_t)(tt - (long)bh * tiles_per_head) * kBtT +
                             tid;
            qi_next = perm_q[p];
            ki_next = perm_k[p];
        }
    };
    auto stage_rows = [&](long tt) {
        if (tid < kBtT) {
            const int bh = (int)(tt / tiles_per_head);
            const size_t hb = (size_t)bh * N;
            int qi = qi_next, ki = ki_next;
            // entries outside [0, N) are recorded and read as row 0
            if (qi < 0 || qi >= N) {
                report(status, kDevPermRange, 10, bh, qi);
                qi = 0;
            }
            if (ki < 0 || ki >= N) {
                report(status, kDevPermRange, 11, bh, ki);
                ki = 0;
            }
            qrow2[tt & 1][tid] = (int)(hb + qi);
            krow2[tt & 1][tid] = (int)(hb + ki);
        }
    };
    // Q, K of tile tt into the buffers of parity tt & 1, and the head's
    // planes below K when that buffer holds another head's
    int planes_h0 = -1, planes_h1 = -1;  // head of each buffer's planes
    auto load_qk = [&](long tt) {
        const int *qr = qrow2[tt & 1], *kr = krow2[tt & 1];
        const uint32_t q_s = base + (uint32_t)(tt & 1) * kQKW;
        const uint32_t k_s = q_s + 16384;
        for (int i = tid; i < kBtT * 8; i += kBtThreads) {
            const int rr = i >> 3, c = i & 7;
            cp_async16(q_s + panel_offset(rr, c, kBtT),
                       qx + (size_t)qr[rr] * d + c * 8);
            cp_async16(k_s + panel_offset(rr, c, NR),
                       kx + (size_t)kr[rr] * d + c * 8);
        }
        const int hh = (int)(tt / tiles_per_head) % H;
        int &ph = (tt & 1) ? planes_h1 : planes_h0;
        if (ph != hh) {
            for (int i = tid; i < Lg_pad * 8; i += kBtThreads) {
                const int rr = i >> 3, c = i & 7;
                cp_async16(k_s + panel_offset(kBtT + rr, c, NR),
                           w_bf16 + ((size_t)hh * Lg_pad + rr) * d + c * 8);
            }
            ph = hh;
        }
    };
    auto load_sums = [&](int bh) {  // the head's B summary (bf16) and A
        for (int i = tid; i < r * 8; i += kBtThreads) {
            const int rr = i >> 3, c = i & 7;
            cp_async16(sB + panel_offset(rr, c, r),
                       Bh + ((size_t)bh * r + rr) * d + c * 8);
        }
        for (int i = tid; i < r / 4; i += kBtThreads)
            cp_async16(sAo + 16 * i, Ag + (size_t)bh * r + 4 * i);
    };
    auto load_g = [&](long tt) {
        const int *qr = qrow2[tt & 1];
        for (int i = tid; i < kBtT * 8; i += kBtThreads) {
            const int rr = i >> 3, c = i & 7;
            cp_async16(sG + panel_offset(rr, c, kBtT),
                       gx + (size_t)qr[rr] * d + c * 8);
        }
    };
    auto load_v = [&](long tt) {
        const int *kr = krow2[tt & 1];
        for (int i = tid; i < kBtT * 8; i += kBtThreads) {
            const int rr = i >> 3, c = i & 7;
            cp_async16(sV + panel_offset(rr, c, kBtT),
                       vx + (size_t)kr[rr] * d + c * 8);
        }
    };
    if (t_begin < t_end) {
        fetch_rows(t_begin);
        stage_rows(t_begin);
        if (t_begin + 1 < t_end) fetch_rows(t_begin + 1);
        __syncthreads();
        load_qk(t_begin);
        load_v(t_begin);
        load_sums((int)(t_begin / tiles_per_head));
        cp_async_commit();
        load_g(t_begin);
    }
    cp_async_commit();

    bool ok = true;
    for (long tt = t_begin; tt < t_end && ok; ++tt) {
        const int bh = (int)(tt / tiles_per_head);
        const uint32_t sQ = base + (uint32_t)(tt & 1) * kQKW;
        const uint32_t sKW = sQ + 16384;  // [NR x 64]: K, then W
        const int *qrow_s = qrow2[tt & 1], *krow_s = krow2[tt & 1];
        const bool more = tt + 1 < t_end;
        // ---------------------------------------------------- phase 0: load
        cp_async_wait<1>();  // all but this tile's dO
        if (more) stage_rows(tt + 1);  // the next tile's rows, parity flips
        if (tt + 2 < t_end) fetch_rows(tt + 2);
        fence_proxy_async_smem();
        __syncthreads();

        // ------------------------------------- phase 1: scores, projections
        if (tid == 0) {
            tc_fence_after();
            const uint32_t id = idesc_bf16(128, NR, false, false);
#pragma unroll
            for (int k = 0; k < d / 16; ++k)
                mma_ss(tm + kCS, smem_desc(sQ + k * 32, 16, 1024),
                       smem_desc(sKW + k * 32, 16, 1024), id, k > 0);
            mma_commit(&mma_bar);
        }
        if (more) load_qk(tt + 1);  // the other parity's readers are done
        cp_async_commit();
        if (!(ok = mma_wait(&mma_bar, mph, 80))) break;

        // ---------------------- phase 2: E on the query's own block, phi, Den
        const int blk = row >> 6;
        const int c0 = 64 * blk + 32 * half;  // this thread's 32 key columns
        float e[32];
        {
            uint32_t v[32];
            tmem_ld32(tm + lane + kCS + c0, v);
            tmem_wait_ld();
            float mx = -INFINITY;
#pragma unroll
            for (int j = 0; j < 32; ++j) {
                e[j] = __uint_as_float(v[j]) * scale;
                mx = fmaxf(mx, e[j]);
            }
            xa[half][row] = mx;
        }
        __syncthreads();
        const float M = fmaxf(xa[0][row], xa[1][row]);
        float lp = 0.0f;
#pragma unroll
        for (int j = 0; j < 32; ++j) {
            e[j] = __expf(e[j] - M);
            lp += e[j];
        }
        xb[half][row] = lp;
        // E rows (bf16), zeros on the other block's keys
#pragma unroll
        for (int q = 0; q < 4; ++q) st8(sE, row, (c0 >> 3) + q, kBtT, e + 8 * q);
        {
            const float z[8] = {0, 0, 0, 0, 0, 0, 0, 0};
            const int cz = 64 * (1 - blk) + 32 * half;
#pragma unroll
            for (int q = 0; q < 4; ++q) st8(sE, row, (cz >> 3) + q, kBtT, z);
        }
        // RACE features of this half's tables
        float u[2 * L > 16 ? 16 : 2 * L];  // projections of TL tables
        {
            uint32_t v[32];
            tmem_ld32(tm + lane + kCS + kBtT, v);  // all Lg_pad projections
            tmem_wait_ld();
#pragma unroll
            for (int b = 0; b < TL * G; ++b)
                u[b] = __uint_as_float(v[half * TL * G + b]);
        }
        float denp = 0.0f;
#pragma unroll
        for (int t = 0; t < TL; ++t) {
            float sp[G], sn[G], phi[R];
#pragma unroll
            for (int b = 0; b < G; ++b) {
                float tu;
                bit_factors_fast(u[t * G + b], beta, sp[b], sn[b], tu);
            }
#pragma unroll
            for (int rr = 0; rr < R; ++rr) {
                float p = 1.0f;
#pragma unroll
                for (int b = 0; b < G; ++b) p *= ((rr >> b) & 1) ? sp[b] : sn[b];
                phi[rr] = p;
            }
            const int tg = half * TL + t;
            float at[R];
            load_table16(Asm + tg * R, at);
#pragma unroll
            for (int rr = 0; rr < R; ++rr) denp = fmaf(phi[rr], at[rr], denp);
            st8(sPhi, row, tg * 2, kBtT, phi);
            st8(sPhi, row, tg * 2 + 1, kBtT, phi + 8);
        }
        xc[half][row] = denp;
        fence_proxy_async_smem();
        tc_fence_before();
        __syncthreads();
        const float lsum = xb[0][row] + xb[1][row];
        const float Den = (xc[0][row] + xc[1][row]) * (1.0f / (float)L);

        // ------------------------------------------- phase 3: E V and phi B
        if (tid == 0) {
            tc_fence_after();
            const uint32_t id = idesc_bf16(128, d, false, true);
#pragma unroll
            for (int k = 0; k < kBtT / 16; ++k)
                mma_ss(tm + kCO,
                       smem_desc(sE + (k >> 2) * 16384 + (k & 3) * 32, 16,
                                 1024),
                       smem_desc(sV + k * 2048, 16384, 1024), id, k > 0);
#pragma unroll
            for (int k = 0; k < r / 16; ++k)
                mma_ss(tm + kCN,
                       smem_desc(sPhi + (k >> 2) * 16384 + (k & 3) * 32, 16,
                                 1024),
                       smem_desc(sB + k * 2048, (uint32_t)r * 128, 1024), id,
                       k > 0);
        }
        cp_async_wait<1>();  // this tile's dO (the barrier below shares it)
        if (!(ok = mma_done(81))) break;

        // ------------------------------------- phase 4: per-query scalars
        const int qrow = qrow_s[row];
        float gv[32], Y[32], Nm[32];
        {
            uint32_t v[32];
            tmem_ld32(tm + lane + kCO + 32 * half, v);
            tmem_wait_ld();
#pragma unroll
            for (int j = 0; j < 32; ++j) Y[j] = __uint_as_float(v[j]);
            tmem_ld32(tm + lane + kCN + 32 * half, v);
            tmem_wait_ld();
#pragma unroll
            for (int j = 0; j < 32; ++j) Nm[j] = __uint_as_float(v[j]);
        }
#pragma unroll
        for (int q = 0; q < 4; ++q) ld8(sG, row, 4 * half + q, kBtT, gv + 8 * q);
        float go = 0.0f, gn = 0.0f;
#pragma unroll
        for (int j = 0; j < 32; ++j) {
            go = fmaf(gv[j], Y[j], go);
            gn = fmaf(gv[j], Nm[j], gn);
        }
        // the two halves' partial dot products (xa is free again: M was
        // read before the last barrier)
        xa[half][row] = go;
        xc[half][row] = gn;
        __syncthreads();
        const float lsE = lsum + eps * __expf(-M);  // (d_s + eps) e^-M
        const float GOs = (xa[0][row] + xa[1][row]) / lsE;
        // G . O_lr with O_lr = (phi B / L) / (Den + eps)
        const float GOlr = (xc[0][row] + xc[1][row]) /
                           ((float)L * (Den + eps));
        const size_t tok = (size_t)qrow;
        const float lam = lambda_tok ? lambda_tok[tok] : lambda;
        const float gs = gates ? gates[2 * tok] : 1.0f;
        const float gl = gates ? gates[2 * tok + 1] : 1.0f;
        const float logds = M + __logf(lsum);
        const float cc = lam * Den + eps;
        const float logD = lse2f(logds, __logf(cc));
        const float m = mode == 1 ? 1.0f : __expf(logds - logD);
        const float invD = __expf(-logD);
        const float dm = mode == 1 ? 0.0f : gs * GOs;
        const float cx = gs * m / lsE;
        const float gdsE = -(gs * m * GOs) / lsE + dm * (cc * invD) * (m / lsum);
        const float cn = gl / (Den + eps);
        const float gDen = -(gl * GOlr) / (Den + eps) - dm * lam * m * invD;
        if (half == 0) {
            if (d_gates) {
                d_gates[2 * tok] = m * GOs;
                d_gates[2 * tok + 1] = GOlr;
            }
            if (d_lambda) d_lambda[tok] = -dm * m * Den * invD;
        }
        {  // dL/dDen repeated over the 16 columns after gNum
            float gd[8];
#pragma unroll
            for (int j = 0; j < 8; ++j) gd[j] = gDen;
            st8(sDU, row, half, kBtT, gd);
        }
        {
            float xv[32], nv[32];
#pragma unroll
            for (int j = 0; j < 32; ++j) {
                xv[j] = cx * gv[j];
                nv[j] = cn * gv[j];
            }
#pragma unroll
            for (int q = 0; q < 4; ++q) {  // X over the dO this thread read
                st8(sG, row, 4 * half + q, kBtT, xv + 8 * q);
                st8(sGN, row, 4 * half + q, kBtT, nv + 8 * q);
            }
        }
        fence_proxy_async_smem();
        tc_fence_before();
        __syncthreads();

        // ------------- phase 5: E^T X, X V^T, gNum B^T, phi^T [gNum | gDen]
        const bool seg_first = tt == t_begin || (tt % tiles_per_head) == 0;
        const bool seg_last =
            tt + 1 == t_end || ((tt + 1) % tiles_per_head) == 0;
        if (tid == 0) {
            tc_fence_after();
            const uint32_t id_p = idesc_bf16(128, kBtT, false, false);
#pragma unroll
            for (int k = 0; k < d / 16; ++k)  // P = X V^T (K = d)
                mma_ss(tm + kCS, smem_desc(sG + k * 32, 16, 1024),
                       smem_desc(sV + k * 32, 16, 1024), id_p, k > 0);
            const uint32_t id_g = idesc_bf16(128, r, false, false);
#pragma unroll
            for (int k = 0; k < d / 16; ++k)  // Gphi = gNum B^T (K = d)
                mma_ss(tm + kCG, smem_desc(sGN + k * 32, 16, 1024),
                       smem_desc(sB + k * 32, 16, 1024), id_g, k > 0);
            mma_commit(&mma_bar);
            // dV and the bucket sums run beside phase 6, which writes
            // none of their operands before it waits for them
            const uint32_t id_v = idesc_bf16(128, d, true, true);
#pragma unroll
            for (int k = 0; k < kBtT / 16; ++k)  // dV = E^T X (K = queries)
                mma_ss(tm + kCdV, smem_desc(sE + k * 2048, 16384, 1024),
                       smem_desc(sG + k * 2048, 16384, 1024), id_v, k > 0);
            // bucket sums (K = queries; M = 128 buckets, rows past r unused;
            // the B operand is gNum followed by the dL/dDen panel)
            const uint32_t id_s = idesc_bf16(128, d + 16, true, true);
#pragma unroll
            for (int k = 0; k < kBtT / 16; ++k)
                mma_ss(tm + kCAcc, smem_desc(sPhi + k * 2048, 16384, 1024),
                       smem_desc(sGN + k * 2048, 16384, 1024), id_s,
                       (k > 0 || !seg_first) ? 1u : 0u);
            mma_commit(&sums_bar);
        }
        if (!(ok = mma_wait(&mma_bar, mph, 82))) break;
        if (more) load_v(tt + 1);  // V's last reader (P = X V^T) is done
        cp_async_commit();

        // ------------- phase 6: dZ, back through the features, dV stores
        float dz[32];  // into sE once dV = E^T X is done
        {
            uint32_t v[32];
            tmem_ld32(tm + lane + kCS + c0, v);
            tmem_wait_ld();
#pragma unroll
            for (int j = 0; j < 32; ++j)
                dz[j] = scale * e[j] * (__uint_as_float(v[j]) + gdsE);
        }
        {
            float du[2 * L > 16 ? 16 : 2 * L];
#pragma unroll
            for (int t = 0; t < TL; ++t) {
                const int tg = half * TL + t;
                uint32_t v[16];
                tmem_ld16(tm + lane + kCG + tg * R, v);
                tmem_wait_ld();
                float sp[G], sn[G], uu[G], phi[R], gp[R];
#pragma unroll
                for (int b = 0; b < G; ++b) {
                    bit_factors_fast(u[t * G + b], beta, sp[b], sn[b],
                                     uu[b]);
                }
                float s = 0.0f, at[R];
                load_table16(Asm + tg * R, at);
#pragma unroll
                for (int rr = 0; rr < R; ++rr) {
                    float p = 1.0f;
#pragma unroll
                    for (int b = 0; b < G; ++b)
                        p *= ((rr >> b) & 1) ? sp[b] : sn[b];
                    phi[rr] = p;
                    gp[rr] = (__uint_as_float(v[rr]) + at[rr] * gDen) *
                             (1.0f / (float)L);
                    s = fmaf(p, gp[rr], s);
                }
#pragma unroll
                for (int b = 0; b < G; ++b) {
                    float g = 0.0f;
#pragma unroll
                    for (int rr = 0; rr < R; ++rr) {
                        const float ga = phi[rr] * (gp[rr] - s);
                        g += ((rr >> b) & 1) ? ga : -ga;
                    }
                    du[t * G + b] = (1.0f - uu[b] * uu[b]) * beta * g;
                }
            }
#pragma unroll
            for (int q = 0; q < TL * G / 8; ++q)
                st8(sDU, row, 4 + (half * TL * G) / 8 + q, kBtT, du + 8 * q);
        }
        // dV and the bucket sums read sE, sG, sPhi, sGN and the dL/dDen
        // columns of sDU
        if (!(ok = mma_wait(&sums_bar, sph, 86))) break;
#pragma unroll
        for (int q = 0; q < 4; ++q) st8(sE, row, (c0 >> 3) + q, kBtT, dz + 8 * q);
        if (seg_last && row < r) {  // this CTA's share of the head's sums
            const long j = (long)blockIdx.x -
                           range_owner((long)bh * tiles_per_head, total_tiles,
                                      gridDim.x);
            float *out =
                part + ((size_t)bh * S_seg + j) * ((size_t)r * d + r);
            uint32_t v[32];
            tmem_ld32(tm + lane + kCAcc + 32 * half, v);
            tmem_wait_ld();
            float4 *o4 =
                reinterpret_cast<float4 *>(out + (size_t)row * d + 32 * half);
#pragma unroll
            for (int q = 0; q < 8; ++q)
                o4[q] = make_float4(__uint_as_float(v[4 * q]),
                                    __uint_as_float(v[4 * q + 1]),
                                    __uint_as_float(v[4 * q + 2]),
                                    __uint_as_float(v[4 * q + 3]));
            if (half == 0) {
                uint32_t a16[16];
                tmem_ld16(tm + lane + kCAcc + d, a16);
                tmem_wait_ld();
                out[(size_t)r * d + row] = __uint_as_float(a16[0]);
            }
        }

        {  // dV staged in sG, sGN (their last readers are done)
            uint32_t v[32];
            tmem_ld32(tm + lane + kCdV + 32 * half, v);
            tmem_wait_ld();
            stage_f32(sG, v);
        }
        fence_proxy_async_smem();
        tc_fence_before();
        __syncthreads();

        // -------------------------- phase 7: dQ = dZ K + dU W, dK = dZ^T Q
        if (tid == 0) {
            tc_fence_after();
            const uint32_t id_q = idesc_bf16(128, d, false, true);
#pragma unroll
            for (int k = 0; k < kBtT / 16; ++k)  // K = keys
                mma_ss(tm + kCO,
                       smem_desc(sE + (k >> 2) * 16384 + (k & 3) * 32, 16,
                                 1024),
                       smem_desc(sKW + k * 2048, (uint32_t)NR * 128, 1024),
                       id_q, k > 0);
#pragma unroll
            for (int k = 0; k < Lg_pad / 16; ++k)  // K = projections
                mma_ss(tm + kCO, smem_desc(sDU + 64 + k * 32, 16, 1024),
                       smem_desc(sKW + kBtT * 128 + k * 2048,
                                 (uint32_t)NR * 128, 1024),
                       id_q, 1);
            const uint32_t id_k = idesc_bf16(128, d, true, true);
#pragma unroll
            for (int k = 0; k < kBtT / 16; ++k)  // K = queries
                mma_ss(tm + kCN, smem_desc(sE + k * 2048, 16384, 1024),
                       smem_desc(sQ + k * 2048, 16384, 1024), id_k, k > 0);
            mma_commit(&mma_bar);
        }
        flush_f32(sG, dv, krow_s);  // beside the MMAs, which do not read sG
        // a new head's B and A: their last readers (Gphi, phase 6) are done
        if (more && (tt + 1) / tiles_per_head != bh)
            load_sums((int)((tt + 1) / tiles_per_head));
        cp_async_commit();
        if (!(ok = mma_wait(&mma_bar, mph, 83))) break;
        if (more) load_g(tt + 1);  // dV's rows have left sG
        cp_async_commit();

        // ------------------------------------------- phase 8: dQ, dK stores
        {  // dQ staged in sE, dK over this tile's Q and K rows (phase 7's
           // MMAs are done; the planes after K stay)
            uint32_t v[32];
            tmem_ld32(tm + lane + kCO + 32 * half, v);
            tmem_wait_ld();
            stage_f32(sE, v);
            tmem_ld32(tm + lane + kCN + 32 * half, v);
            tmem_wait_ld();
            stage_f32(sQ, v);
        }
        tc_fence_before();
        __syncthreads();
        flush_f32(sE, dq, qrow_s);
        flush_f32(sQ, dk, krow_s);
        __syncthreads();  // TMEM and shared memory are reused by the next tile
    }
    cp_async_wait<0>();
    tc_fence_before();
    __syncthreads();
    if (warp == 0) tmem_dealloc(tm, 512);
}

// RACE key side of the backward on tensor cores, per 128-key tile (keys in
// their original order): with gB = sum_i phi(Q_i) gNum_i^T / L and
// gA = sum_i phi(Q_i) dL/dDen_i / L (bf16 / fp32, per head; summed from the
// block kernel's partials, in CTA order, whenever a CTA starts on a head),
//   MMA  U = K W^T                         projections
//   CUDA phi(K)
//   MMA  dV_k = phi gB,  Gphi = V gB^T
//   CUDA dV += dV_k; dL/dphi = Gphi + gA, back through the corner softmax
//        and tanh -> dL/d(W k)
//   MMA  dK_k = dL/d(W k) W
//   CUDA dK += dK_k
// Each key belongs to one tile: plain read-modify-write of dV and dK (the
// sparse parts were stored by the block kernel before). A tile's 128 keys
// are consecutive rows, so K, V and the old dV, dK rows arrive by TMA (the
// fp32 rows as two boxes of 32 columns in the 128-byte swizzle) and the
// updated dV, dK rows leave by TMA stores from the same boxes.
constexpr uint32_t kKU = 0;     // projections [0, 32)
constexpr uint32_t kKdV = 32;   // phi gB
constexpr uint32_t kKG = 96;    // V gB^T (r <= 128)
constexpr uint32_t kKdK = 224;  // dL/du W

template <int L>
__global__ void __launch_bounds__(kBtThreads, 1)
    k_bwd_keys_tc(const __grid_constant__ CUtensorMap tmK,
                  const __grid_constant__ CUtensorMap tmV,
                  const __grid_constant__ CUtensorMap tmDK,
                  const __grid_constant__ CUtensorMap tmDV,
                  const uint16_t *__restrict__ w_bf16,
                  const float *__restrict__ part, int S_seg, int blk_grid,
                  int N, int H, float beta, int tiles_per_head,
                  long total_tiles, DeviceStatus *status) {
    constexpr int R = 16, G = 4;
    constexpr int r = L * R, Lg = L * G;
    constexpr int Lg_pad = (Lg + 15) / 16 * 16;
    constexpr int NR = kBtT + Lg_pad;
    constexpr int TL = L / 2;
    constexpr int d = kBtD;
    extern __shared__ unsigned char smem_raw[];
    __shared__ uint64_t mma_bar, k_bar, v_bar, old_bar;
    __shared__ uint32_t tbase;
    __shared__ int abort_flag;
    volatile int *abort = &abort_flag;
    const int tid = threadIdx.x, warp = tid >> 5, lane_id = tid & 31;
    const int half = warp >> 2;
    const int row = (warp & 3) * 32 + lane_id;  // key of the tile = lane
    const uint32_t lane = (uint32_t)((warp & 3) * 32) << 16;

    const uint32_t base = align1k(smem_u32(smem_raw));
    const uint32_t sKW = base;                        // [NR x 64]: K, W
    const uint32_t sV = sKW + align1k(NR * 128);      // [128 x 64]
    const uint32_t sPhi = sV + 16384;                 // [128 x r]
    const uint32_t sgB = sPhi + align1k(kBtT * r * 2);  // [r x 64]
    const uint32_t sDU = sgB + align1k(r * 128);      // [128 x 64]
    // fp32 dV, dK rows of the tile as the block kernel left them: per
    // matrix two boxes [128 x 32] of 128-byte rows, the 16-byte chunk c of
    // row j at chunk c ^ (j & 7)
    const uint32_t sDVo = sDU + 16384;
    const uint32_t sDKo = sDVo + 32768;
    const uint32_t sAo = sDKo + 32768;                 // fp32 gA [r]
    float *gAs = reinterpret_cast<float *>(smem_raw + (sAo - smem_u32(smem_raw)));

    const long t_begin = total_tiles * blockIdx.x / gridDim.x;
    const long t_end = total_tiles * (blockIdx.x + 1) / gridDim.x;
    if (warp == 0) tmem_alloc(&tbase, 512);
    if (tid == 0) {
        mbar_init(&mma_bar, 1);
        mbar_init(&k_bar, 1);
        mbar_init(&v_bar, 1);
        mbar_init(&old_bar, 1);
        abort_flag = 0;
        fence_mbar_init();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tm = tbase;
    uint32_t mph = 0;
    // every thread waits for a copy barrier; all leave if any wait ran out
    auto copy_wait = [&](uint64_t *bar, long tt, int site) -> bool {
        const bool ok = mbar_wait_or_abort(bar, (uint32_t)(tt - t_begin) & 1,
                                           abort, status, site);
        return __syncthreads_and(ok);
    };
    auto mma_done = [&](int site) -> bool {
        if (tid == 0) mma_commit(&mma_bar);
        const bool ok = mbar_wait_or_abort(&mma_bar, mph & 1, abort, status,
                                           site);
        ++mph;
        tc_fence_after();
        return __syncthreads_and(ok);
    };
    auto st8 = [&](uint32_t region, int rr, int chunk, int rows,
                   const float *v) {
        st_shared_bf16x8(region + panel_offset(rr, chunk, rows), v);
    };
    // this thread's 32 TMEM columns (box `half`) added into its old row
    auto add_old = [&](uint32_t region, const uint32_t *v) {
        const uint32_t rb = region + 16384u * half + (uint32_t)row * 128;
#pragma unroll
        for (int q = 0; q < 8; ++q) {
            const uint32_t a16 = rb + ((uint32_t)(q ^ (row & 7)) << 4);
            const uint4 a = ld_shared_v4(a16);
            st_shared_v4(a16,
                         __float_as_uint(__uint_as_float(a.x) +
                                         __uint_as_float(v[4 * q])),
                         __float_as_uint(__uint_as_float(a.y) +
                                         __uint_as_float(v[4 * q + 1])),
                         __float_as_uint(__uint_as_float(a.z) +
                                         __uint_as_float(v[4 * q + 2])),
                         __float_as_uint(__uint_as_float(a.w) +
                                         __uint_as_float(v[4 * q + 3])));
        }
    };
    auto tile_row0 = [&](long tt) {
        const int bh = (int)(tt / tiles_per_head);
        return (size_t)bh * N +
               (size_t)(tt - (long)bh * tiles_per_head) * kBtT;
    };
    // thread 0 issues every TMA copy; the last tile a copy was issued for,
    // per barrier, lets an aborted CTA drain its copies before it exits
    long k_last = -1, v_last = -1, old_last = -1;
    auto load_k = [&](long tt) {
        mbar_expect_tx(&k_bar, 16384);
        tma_load_2d(sKW, &tmK, 0, (int)tile_row0(tt), &k_bar);
        k_last = tt;
    };
    auto load_v = [&](long tt) {
        mbar_expect_tx(&v_bar, 16384);
        tma_load_2d(sV, &tmV, 0, (int)tile_row0(tt), &v_bar);
        v_last = tt;
    };
    if (tid == 0 && t_begin < t_end) {
        load_k(t_begin);
        load_v(t_begin);
    }

    int cur_bh = -1;
    bool ok = true;
    for (long tt = t_begin; tt < t_end && ok; ++tt) {
        const int bh = (int)(tt / tiles_per_head);
        const int h = bh % H;
        const size_t row0 = tile_row0(tt);
        const bool new_head = bh != cur_bh;
        if (new_head) {  // the head's planes, gB (bf16) and gA
            for (int i = tid; i < Lg_pad * 8; i += kBtThreads) {
                const int rr = i >> 3, c = i & 7;
                cp_async16(sKW + panel_offset(kBtT + rr, c, NR),
                           w_bf16 + ((size_t)h * Lg_pad + rr) * d + c * 8);
            }
            // gB (bf16 panel) and gA: the block kernel's partials of the
            // CTAs that worked on the head, summed in CTA order, times 1 / L
            const size_t per = (size_t)r * d + r;
            const float *p0 = part + (size_t)bh * S_seg * per;
            const int nparts =
                (int)(range_owner((long)(bh + 1) * tiles_per_head - 1,
                                  total_tiles, blk_grid) -
                      range_owner((long)bh * tiles_per_head, total_tiles,
                                  blk_grid) +
                      1);
            // each thread: NC 16-byte chunks of gB (8 values each) and at
            // most one entry of gA, all of one partial's loads in flight at
            // once, partials in CTA order
            constexpr int NC = r * 8 / kBtThreads;
            static_assert(NC * kBtThreads == r * 8 && r <= kBtThreads,
                          "gB chunks and gA entries spread evenly");
            const float inv = 1.0f / (float)L;
            float sum[NC][8] = {};
            float sa = 0.f;
            for (int j = 0; j < nparts; ++j) {
                const float *pj = p0 + (size_t)j * per;
                float4 a[NC], b2[NC];
#pragma unroll
                for (int q = 0; q < NC; ++q) {
                    const int i = tid + q * kBtThreads;
                    const float4 *src = reinterpret_cast<const float4 *>(
                        pj + (size_t)(i >> 3) * d + (i & 7) * 8);
                    a[q] = src[0];
                    b2[q] = src[1];
                }
                const float av = tid < r ? pj[(size_t)r * d + tid] : 0.f;
#pragma unroll
                for (int q = 0; q < NC; ++q) {
                    sum[q][0] += a[q].x;
                    sum[q][1] += a[q].y;
                    sum[q][2] += a[q].z;
                    sum[q][3] += a[q].w;
                    sum[q][4] += b2[q].x;
                    sum[q][5] += b2[q].y;
                    sum[q][6] += b2[q].z;
                    sum[q][7] += b2[q].w;
                }
                sa += av;
            }
#pragma unroll
            for (int q = 0; q < NC; ++q) {
                const int i = tid + q * kBtThreads;
#pragma unroll
                for (int e = 0; e < 8; ++e) sum[q][e] *= inv;
                st8(sgB, i >> 3, i & 7, r, sum[q]);
            }
            if (tid < r) gAs[tid] = sa * inv;
            cp_async_commit();
            cur_bh = bh;
        }
        if (tid == 0) {  // old dV, dK rows of this tile (read back later)
            bulk_wait_read();  // the last tile's stores have read the boxes
            mbar_expect_tx(&old_bar, 65536);
            const int y = (int)row0;
            tma_load_2d(sDVo, &tmDV, 0, y, &old_bar);
            tma_load_2d(sDVo + 16384, &tmDV, 32, y, &old_bar);
            tma_load_2d(sDKo, &tmDK, 0, y, &old_bar);
            tma_load_2d(sDKo + 16384, &tmDK, 32, y, &old_bar);
            old_last = tt;
        }
        cp_async_wait<0>();  // planes, gB, gA on a head change
        fence_proxy_async_smem();
        if (!(ok = copy_wait(&k_bar, tt, 93))) break;  // K of this tile

        // projections U = K W^T
        if (tid == 0) {
            tc_fence_after();
            const uint32_t id = idesc_bf16(128, Lg_pad, false, false);
#pragma unroll
            for (int k = 0; k < d / 16; ++k)
                mma_ss(tm + kKU, smem_desc(sKW + k * 32, 16, 1024),
                       smem_desc(sKW + kBtT * 128 + k * 32, 16, 1024), id,
                       k > 0);
        }
        if (!(ok = mma_done(90))) break;
        if (tid == 0 && tt + 1 < t_end) load_k(tt + 1);  // K is consumed

        // features of this half's tables
        float u[2 * L > 16 ? 16 : 2 * L];
        {
            uint32_t v[32];
            tmem_ld32(tm + lane + kKU, v);
            tmem_wait_ld();
#pragma unroll
            for (int b = 0; b < TL * G; ++b)
                u[b] = __uint_as_float(v[half * TL * G + b]);
        }
#pragma unroll
        for (int t = 0; t < TL; ++t) {
            float sp[G], sn[G], phi[R];
#pragma unroll
            for (int b = 0; b < G; ++b) {
                float tu;
                bit_factors_fast(u[t * G + b], beta, sp[b], sn[b], tu);
            }
#pragma unroll
            for (int rr = 0; rr < R; ++rr) {
                float p = 1.0f;
#pragma unroll
                for (int b = 0; b < G; ++b) p *= ((rr >> b) & 1) ? sp[b] : sn[b];
                phi[rr] = p;
            }
            const int tg = half * TL + t;
            st8(sPhi, row, tg * 2, kBtT, phi);
            st8(sPhi, row, tg * 2 + 1, kBtT, phi + 8);
        }
        fence_proxy_async_smem();
        tc_fence_before();
        if (!(ok = copy_wait(&v_bar, tt, 94))) break;  // V of this tile

        // dV_k = phi gB, Gphi = V gB^T
        if (tid == 0) {
            tc_fence_after();
            const uint32_t id_v = idesc_bf16(128, d, false, true);
#pragma unroll
            for (int k = 0; k < r / 16; ++k)
                mma_ss(tm + kKdV,
                       smem_desc(sPhi + (k >> 2) * 16384 + (k & 3) * 32, 16,
                                 1024),
                       smem_desc(sgB + k * 2048, (uint32_t)r * 128, 1024),
                       id_v, k > 0);
            const uint32_t id_g = idesc_bf16(128, r, false, false);
#pragma unroll
            for (int k = 0; k < d / 16; ++k)
                mma_ss(tm + kKG, smem_desc(sV + k * 32, 16, 1024),
                       smem_desc(sgB + k * 32, 16, 1024), id_g, k > 0);
        }
        if (!(ok = mma_done(91))) break;
        if (tid == 0 && tt + 1 < t_end) load_v(tt + 1);  // V is consumed
        if (!(ok = copy_wait(&old_bar, tt, 95))) break;

        {
            uint32_t v[32];
            tmem_ld32(tm + lane + kKdV + 32 * half, v);
            tmem_wait_ld();
            add_old(sDVo, v);
        }
        {
            float du[2 * L > 16 ? 16 : 2 * L];
#pragma unroll
            for (int t = 0; t < TL; ++t) {
                const int tg = half * TL + t;
                uint32_t v[16];
                tmem_ld16(tm + lane + kKG + tg * R, v);
                tmem_wait_ld();
                float sp[G], sn[G], uu[G], phi[R], gp[R];
#pragma unroll
                for (int b = 0; b < G; ++b) {
                    bit_factors_fast(u[t * G + b], beta, sp[b], sn[b],
                                     uu[b]);
                }
                float s = 0.0f, at[R];
                load_table16(gAs + tg * R, at);
#pragma unroll
                for (int rr = 0; rr < R; ++rr) {
                    float p = 1.0f;
#pragma unroll
                    for (int b = 0; b < G; ++b)
                        p *= ((rr >> b) & 1) ? sp[b] : sn[b];
                    phi[rr] = p;
                    gp[rr] = __uint_as_float(v[rr]) + at[rr];
                    s = fmaf(p, gp[rr], s);
                }
#pragma unroll
                for (int b = 0; b < G; ++b) {
                    float g = 0.0f;
#pragma unroll
                    for (int rr = 0; rr < R; ++rr) {
                        const float ga = phi[rr] * (gp[rr] - s);
                        g += ((rr >> b) & 1) ? ga : -ga;
                    }
                    du[t * G + b] = (1.0f - uu[b] * uu[b]) * beta * g;
                }
            }
#pragma unroll
            for (int q = 0; q < TL * G / 8; ++q)
                st8(sDU, row, (half * TL * G) / 8 + q, kBtT, du + 8 * q);
        }
        fence_proxy_async_smem();  // the dV sums, for the TMA store
        tc_fence_before();
        __syncthreads();

        // dK_k = dL/du W
        if (tid == 0) {
            tma_store_2d(&tmDV, 0, (int)row0, sDVo);
            tma_store_2d(&tmDV, 32, (int)row0, sDVo + 16384);
            bulk_commit();
            tc_fence_after();
            const uint32_t id_q = idesc_bf16(128, d, false, true);
#pragma unroll
            for (int k = 0; k < Lg_pad / 16; ++k)
                mma_ss(tm + kKdK, smem_desc(sDU + k * 32, 16, 1024),
                       smem_desc(sKW + kBtT * 128 + k * 2048,
                                 (uint32_t)NR * 128, 1024),
                       id_q, k > 0);
        }
        if (!(ok = mma_done(92))) break;
        {
            uint32_t v[32];
            tmem_ld32(tm + lane + kKdK + 32 * half, v);
            tmem_wait_ld();
            add_old(sDKo, v);
        }
        fence_proxy_async_smem();
        tc_fence_before();
        __syncthreads();
        if (tid == 0) {
            tma_store_2d(&tmDK, 0, (int)row0, sDKo);
            tma_store_2d(&tmDK, 32, (int)row0, sDKo + 16384);
            bulk_commit();
        }
    }
    cp_async_wait<0>();
    if (tid == 0) {
        if (!ok) {  // an abort: the copies issued last may still be landing
            uint64_t *bars[3] = {&k_bar, &v_bar, &old_bar};
            const long last[3] = {k_last, v_last, old_last};
            for (int i = 0; i < 3; ++i)
                if (last[i] >= 0)
                    mbar_wait(bars[i], (uint32_t)(last[i] - t_begin) & 1,
                              status, 96);
        }
        bulk_wait_all();  // the last stores are complete
    }
    tc_fence_before();
    __syncthreads();
    if (warp == 0) tmem_dealloc(tm, 512);
}

}  // namespace

bool bwd_tc_supported(const Plan &P) {
    return P.dtype == ELSAA_BF16 && P.d == kBtD && P.b == 64 &&
           P.gamma == 4 && (P.L == 4 || P.L == 8) && P.N % kBtT == 0 &&
           P.nb == 0 && (long)P.BH * P.N < (1l << 31);
}

size_t bwd_tc_smem(const Plan &P) {
    const size_t r = (size_t)P.L * 16;
    const size_t lg_pad = ((size_t)P.L * 4 + 15) / 16 * 16;
    auto a1k = [](size_t x) { return (x + 1023) / 1024 * 1024; };
    return 1024 + 2 * (16384 + a1k((kBtT + lg_pad) * 128)) + 16384 * 4 +
           32768 + a1k(kBtT * r * 2) + a1k(r * 128) + r * 4;
}

int bwd_tc_grid(const Plan &P) {
    const long total = (long)(P.N / kBtT) * P.BH;
    return (int)(total < kBtGrid ? total : kBtGrid);
}

int bwd_tc_segments(const Plan &P) {
    const int T = P.N / kBtT;
    const long total = (long)T * P.BH;
    const long grid = bwd_tc_grid(P);
    long most = 1;
    for (long bh = 0; bh < P.BH; ++bh) {
        const long n = range_owner((bh + 1) * T - 1, total, grid) -
                       range_owner(bh * T, total, grid) + 1;
        if (n > most) most = n;
    }
    return (int)most;
}

cudaError_t launch_bwd_block_tc(const Plan &P, const void *q, const void *k,
                                const void *v, const void *d_o,
                                const uint16_t *w_bf16, const uint16_t *Bh,
                                const float *A, const int32_t *perm_q,
                                const int32_t *perm_k, const float *lambda_tok,
                                const float *gates, float *dq, float *dk,
                                float *dv, float *d_gates, float *d_lambda,
                                float *part, DeviceStatus *status,
                                cudaStream_t st) {
    const int tiles_per_head = P.N / kBtT;
    const long total = (long)tiles_per_head * P.BH;
    const int grid = bwd_tc_grid(P);
    const int S_seg = bwd_tc_segments(P);
    const size_t smem = bwd_tc_smem(P);
    auto launch = [&](auto kern) {
        cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             (int)smem);
        kern<<<grid, kBtThreads, smem, st>>>(
            (const uint16_t *)q, (const uint16_t *)k, (const uint16_t *)v,
            (const uint16_t *)d_o, w_bf16, Bh, A, perm_q, perm_k, lambda_tok,
            gates, P.N, P.H, P.beta, P.eps, P.scale, P.lambda, P.fusion_mode,
            tiles_per_head, total, dq, dk, dv, d_gates, d_lambda, part, S_seg,
            status);
        return cudaGetLastError();
    };
    return P.L == 8 ? launch(k_bwd_block_tc<8>) : launch(k_bwd_block_tc<4>);
}

}  // namespace elsaa

namespace elsaa {

size_t bwd_keys_tc_smem(const Plan &P) {
    const size_t r = (size_t)P.L * 16;
    const size_t lg_pad = ((size_t)P.L * 4 + 15) / 16 * 16;
    auto a1k = [](size_t x) { return (x + 1023) / 1024 * 1024; };
    return 1024 + a1k((kBtT + lg_pad) * 128) + 16384 + a1k(kBtT * r * 2) +
           a1k(r * 128) + 16384 + 2 * 32768 + r * 4;
}

cudaError_t launch_bwd_keys_tc(const Plan &P, const void *k, const void *v,
                               const uint16_t *w_bf16, const float *part,
                               float *dk, float *dv, DeviceStatus *status,
                               cudaStream_t st) {
    const int tiles_per_head = P.N / kBtT;
    const long total = (long)tiles_per_head * P.BH;
    int dev = 0, sms = 148;
    if (cudaGetDevice(&dev) == cudaSuccess)
        cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    const int grid = (int)(total < sms ? total : sms);
    const size_t smem = bwd_keys_tc_smem(P);
    const int S_seg = bwd_tc_segments(P), blk_grid = bwd_tc_grid(P);
    const uint64_t rows = (uint64_t)P.BH * P.N;
    CUtensorMap tmK, tmV, tmDK, tmDV;
    cudaError_t e = make_tma_map_bf16(&tmK, k, rows, kBtD, kBtT);
    if (e == cudaSuccess) e = make_tma_map_bf16(&tmV, v, rows, kBtD, kBtT);
    if (e == cudaSuccess)
        e = make_tma_map_f32(&tmDK, dk, rows, kBtD, 32, kBtT);
    if (e == cudaSuccess)
        e = make_tma_map_f32(&tmDV, dv, rows, kBtD, 32, kBtT);
    if (e != cudaSuccess) return e;
    auto launch = [&](auto kern) {
        cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             (int)smem);
        kern<<<grid, kBtThreads, smem, st>>>(tmK, tmV, tmDK, tmDV, w_bf16,
                                             part, S_seg, blk_grid, P.N, P.H,
                                             P.beta, tiles_per_head, total,
                                             status);
        return cudaGetLastError();
    };
    return P.L == 8 ? launch(k_bwd_keys_tc<8>) : launch(k_bwd_keys_tc<4>);
}

}  // namespace elsaa
