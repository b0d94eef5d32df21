// Per-query top-k selector for the sparse branch (selector = 1): a
// selector that Section 3 ("sorted Hamming LSH") names as future work. The
// steps after the hash and the stable sort of Algorithm sortLSH:
//
//   k_topk_sums    block sums of the sorted queries and keys (fp32,
//                  sequential over increasing sorted position)
//   k_topk_cand    block scores s(t, u) = <qbar_t, kbar_u> (canonical fp32
//                  FMA chain) and, per query block, its own key block plus
//                  the c - 1 best other blocks (equal scores: lower u)
//   k_topk_select  per query, the canonical fp32 chain <q_i, k_j> of every
//                  candidate key and a warp radix select of the k best
//                  (equal scores: lower original key index), written as a
//                  bitmask over the candidates
//   k_topk_export  (on request) the selected key indices of each query,
//                  increasing
//
// Every selection decision is taken in the precision of the canonical chain
// acc = fmaf(a[e], b[e], acc), e = 0 .. d - 1 from +0.0f, exactly as the
// sort hash does, so the selected sets are bit-identical to the oracle's.
// The block kernels then run the sparse block step over the candidate keys
// with the unselected ones masked.
#include "device_common.cuh"

namespace elsaa {

namespace {

constexpr int kSelThreads = 256;
constexpr int kSelWarps = kSelThreads / 32;
constexpr int kSelPad = 4;  // fp32 row padding of the staged keys

// Order-preserving map of fp32 scores to uint32 (larger score, larger key).
// -0.0 is taken as +0.0, as the float comparison of the oracle does.
__device__ __forceinline__ uint32_t ordered_key(float f) {
    if (f == 0.0f) f = 0.0f;
    const uint32_t u = __float_as_uint(f);
    return (u & 0x80000000u) ? ~u : (u | 0x80000000u);
}

// Grid (T, BH, 2), d threads: sums[w][bh][t][e] over the sorted positions
// [t b, (t + 1) b) of queries (w = 0) or keys (w = 1).
template <typename X>
__global__ void k_topk_sums(const X *__restrict__ qx, const X *__restrict__ kx,
                            const int32_t *__restrict__ perm_q,
                            const int32_t *__restrict__ perm_k, int N, int d,
                            int b, float *__restrict__ sums,
                            DeviceStatus *status) {
    const int t = blockIdx.x, bh = blockIdx.y, w = blockIdx.z;
    const int T = gridDim.x, BH = gridDim.y, e = threadIdx.x;
    const X *x = (w ? kx : qx) + (size_t)bh * N * d;
    const int32_t *pm = (w ? perm_k : perm_q) + (size_t)bh * N;
    float acc = 0.0f;
    for (int p = t * b; p < (t + 1) * b; ++p) {
        int i = pm[p];
        if (i < 0 || i >= N) {
            if (e == 0) report(status, kDevPermRange, 20, bh, i);
            i = 0;
        }
        acc = __fadd_rn(acc, to_f32<X>(x[(size_t)i * d + e]));
    }
    sums[(((size_t)w * BH + bh) * T + t) * d + e] = acc;
}

// Grid (T, BH), kSelThreads threads; dynamic shared memory: T scores, T
// flags, the block's query sum. cand[bh][t][0 .. c) = t, then the c - 1
// blocks u != t of largest score in order (equal scores: lower u).
__global__ void __launch_bounds__(kSelThreads)
    k_topk_cand(const float *__restrict__ sums, int d, int c,
                int32_t *__restrict__ cand) {
    extern __shared__ float csm[];
    const int t = blockIdx.x, bh = blockIdx.y;
    const int T = gridDim.x, BH = gridDim.y;
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    float *qs = csm;                     // [d]
    float *sc = qs + d;                  // [T]
    int *taken = reinterpret_cast<int *>(sc + T);  // [T]
    __shared__ float bs[kSelWarps];
    __shared__ int bu[kSelWarps];
    const float *qsum = sums + ((size_t)bh * T + t) * d;
    const float *ksum = sums + ((size_t)(BH + bh) * T) * d;
    for (int e = tid; e < d; e += kSelThreads) qs[e] = qsum[e];
    __syncthreads();
    for (int u = tid; u < T; u += kSelThreads) {
        const float *kr = ksum + (size_t)u * d;
        float acc = 0.0f;
        for (int e = 0; e < d; ++e) acc = fmaf(qs[e], kr[e], acc);
        sc[u] = acc;
        taken[u] = u == t;
    }
    __syncthreads();
    int32_t *out = cand + ((size_t)bh * T + t) * c;
    if (tid == 0) out[0] = t;
    for (int m = 1; m < c; ++m) {
        // (score, u) lexicographic best: larger score, then lower u
        float best = 0.0f;
        int bu_ = -1;
        for (int u = tid; u < T; u += kSelThreads)
            if (!taken[u] && (bu_ < 0 || sc[u] > best)) {
                best = sc[u];
                bu_ = u;
            }
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) {
            const float ob = __shfl_xor_sync(0xffffffffu, best, o);
            const int ou = __shfl_xor_sync(0xffffffffu, bu_, o);
            if (ou >= 0 && (bu_ < 0 || ob > best || (ob == best && ou < bu_))) {
                best = ob;
                bu_ = ou;
            }
        }
        if (lane == 0) {
            bs[warp] = best;
            bu[warp] = bu_;
        }
        __syncthreads();
        if (tid == 0) {
            float b0 = 0.0f;
            int u0 = -1;
            for (int w = 0; w < kSelWarps; ++w)
                if (bu[w] >= 0 &&
                    (u0 < 0 || bs[w] > b0 || (bs[w] == b0 && bu[w] < u0))) {
                    b0 = bs[w];
                    u0 = bu[w];
                }
            out[m] = u0;
            if (u0 >= 0) taken[u0] = 1;
        }
        __syncthreads();
    }
}

// Grid (T, BH), kSelThreads threads, M = c b / 32 candidate words (<= 16).
// Dynamic shared memory: the candidate keys as fp32 rows of d + kSelPad,
// their original indices, one query row per warp.
template <typename X, int M>
__global__ void __launch_bounds__(kSelThreads)
    k_topk_select(const X *__restrict__ qx, const X *__restrict__ kx,
                  const int32_t *__restrict__ perm_q,
                  const int32_t *__restrict__ perm_k,
                  const int32_t *__restrict__ cand, int N, int d, int b,
                  int c, int k, uint32_t *__restrict__ selmask,
                  DeviceStatus *status) {
    extern __shared__ __align__(16) float ssm[];
    const int t = blockIdx.x, bh = blockIdx.y, T = gridDim.x;
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int nc = 32 * M, ds = d + kSelPad;
    float *kc = ssm;                                    // [nc][ds]
    int *cidx = reinterpret_cast<int *>(kc + (size_t)nc * ds);  // [nc]
    float *qrow = reinterpret_cast<float *>(cidx + nc) + warp * d;  // [d]
    const X *qh = qx + (size_t)bh * N * d;
    const X *kh = kx + (size_t)bh * N * d;
    const int32_t *pq = perm_q + (size_t)bh * N;
    const int32_t *pk = perm_k + (size_t)bh * N;
    const int32_t *cb = cand + ((size_t)bh * T + t) * c;
    // stage the c b candidate keys (candidate r = key r % b of block r / b)
    for (int r = warp; r < nc; r += kSelWarps) {
        int u = cb[r / b];
        if (u < 0 || u >= T) u = t;
        int j = pk[u * b + r % b];
        if (j < 0 || j >= N) {
            if (lane == 0) report(status, kDevPermRange, 21, bh, j);
            j = 0;
        }
        if (lane == 0) cidx[r] = j;
        for (int e = lane; e < d; e += 32)
            kc[(size_t)r * ds + e] = to_f32<X>(kh[(size_t)j * d + e]);
    }
    __syncthreads();
    const int W = M;  // mask words per query
    for (int qq = warp; qq < b; qq += kSelWarps) {
        const int p = t * b + qq;
        int i = pq[p];
        if (i < 0 || i >= N) {
            if (lane == 0) report(status, kDevPermRange, 22, bh, i);
            i = 0;
        }
        __syncwarp();
        for (int e = lane; e < d; e += 32)
            qrow[e] = to_f32<X>(qh[(size_t)i * d + e]);
        __syncwarp();
        // canonical chains: candidate lane + 32 m, e = 0 .. d - 1 in order
        float acc[M];
#pragma unroll
        for (int m = 0; m < M; ++m) acc[m] = 0.0f;
        for (int e = 0; e < d; e += 4) {
            const float4 qv = *reinterpret_cast<const float4 *>(qrow + e);
#pragma unroll
            for (int m = 0; m < M; ++m) {
                const float4 kv = *reinterpret_cast<const float4 *>(
                    kc + (size_t)(lane + 32 * m) * ds + e);
                acc[m] = fmaf(qv.x, kv.x, acc[m]);
                acc[m] = fmaf(qv.y, kv.y, acc[m]);
                acc[m] = fmaf(qv.z, kv.z, acc[m]);
                acc[m] = fmaf(qv.w, kv.w, acc[m]);
            }
        }
        uint32_t key[M];
#pragma unroll
        for (int m = 0; m < M; ++m) key[m] = ordered_key(acc[m]);
        // the k-th largest key: MSB-first radix select
        uint32_t pre = 0, msk = 0;
        int above = 0;
        for (int bit = 31; bit >= 0; --bit) {
            const uint32_t bm = 1u << bit, want = pre | bm, mk = msk | bm;
            int cnt = 0;
#pragma unroll
            for (int m = 0; m < M; ++m) cnt += (key[m] & mk) == want;
            cnt = __reduce_add_sync(0xffffffffu, cnt);
            if (above + cnt >= k)
                pre = want;
            else
                above += cnt;
            msk = mk;
        }
        // keys equal to the threshold: the need lowest original indices
        const int need = k - above;
        int ties = 0;
#pragma unroll
        for (int m = 0; m < M; ++m) ties += key[m] == pre;
        ties = __reduce_add_sync(0xffffffffu, ties);
        int jmax = 0x7fffffff;
        if (ties > need) {
            uint32_t jp = 0, jm = 0;
            int below = 0;
            for (int bit = 30; bit >= 0; --bit) {
                const uint32_t bm = 1u << bit, mk = jm | bm;
                int cnt = 0;  // ties whose index has this bit clear
#pragma unroll
                for (int m = 0; m < M; ++m)
                    cnt += key[m] == pre &&
                           ((uint32_t)cidx[lane + 32 * m] & mk) == jp;
                cnt = __reduce_add_sync(0xffffffffu, cnt);
                if (below + cnt < need) {
                    below += cnt;
                    jp |= bm;
                }
                jm = mk;
            }
            jmax = (int)jp;
        }
        uint32_t *out = selmask + ((size_t)bh * N + p) * W;
#pragma unroll
        for (int m = 0; m < M; ++m) {
            const bool s = key[m] > pre ||
                           (key[m] == pre && cidx[lane + 32 * m] <= jmax);
            const uint32_t word = __ballot_sync(0xffffffffu, s);
            if (lane == m) out[m] = word;
        }
    }
}

// Grid (ceil(N / 8), BH), kSelThreads threads: one warp per sorted query
// position; out[bh][i][0 .. k) = the selected key indices of query i,
// increasing.
__global__ void __launch_bounds__(kSelThreads)
    k_topk_export(const int32_t *__restrict__ perm_q,
                  const int32_t *__restrict__ perm_k,
                  const int32_t *__restrict__ cand,
                  const uint32_t *__restrict__ selmask, int N, int b, int c,
                  int k, int32_t *__restrict__ out, DeviceStatus *status) {
    __shared__ int list[kSelWarps][512];
    const int bh = blockIdx.y, T = N / b;
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int p = blockIdx.x * kSelWarps + warp;
    if (p >= N) return;  // whole warps
    const int t = p / b, W = c * b / 32;
    const int32_t *pk = perm_k + (size_t)bh * N;
    const int32_t *cb = cand + ((size_t)bh * T + t) * c;
    const uint32_t *mw = selmask + ((size_t)bh * N + p) * W;
    int n = 0;
    for (int m = 0; m < W; ++m) {
        const int r = 32 * m + lane;
        const bool s = (mw[m] >> lane) & 1u;
        const unsigned bal = __ballot_sync(0xffffffffu, s);
        if (s && n + __popc(bal & ((1u << lane) - 1u)) < 512) {
            int u = cb[r / b];
            if (u < 0 || u >= T) u = t;
            list[warp][n + __popc(bal & ((1u << lane) - 1u))] =
                pk[u * b + r % b];
        }
        n += __popc(bal);
    }
    __syncwarp();
    int i = perm_q[(size_t)bh * N + p];
    if (n != k || i < 0 || i >= N) {
        if (lane == 0) report(status, kDevPermRange, 23, bh, n);
        return;
    }
    int32_t *o = out + ((size_t)bh * N + i) * k;
    for (int q = lane; q < n; q += 32) {
        const int v = list[warp][q];
        int rank = 0;
        for (int x = 0; x < n; ++x) rank += list[warp][x] < v;
        o[rank] = v;
    }
}

size_t select_smem(const Plan &P) {
    const int nc = P.tk_c * P.b;
    return (size_t)nc * (P.d + kSelPad) * 4 + (size_t)nc * 4 +
           (size_t)kSelWarps * P.d * 4;
}

}  // namespace

bool topk_supported(const Plan &P, const char **msg) {
    const int nc = P.tk_c * P.b;
    if (nc % 32 != 0 || nc / 32 > 16) {
        *msg = "selector 1: topk_blocks * block_size must be at most 512";
        return false;
    }
    if (P.N / P.b > 8192) {
        *msg = "selector 1: at most 8192 blocks per head";
        return false;
    }
    if (select_smem(P) > 200 * 1024) {
        *msg = "selector 1: the candidate keys of a block (topk_blocks * "
               "block_size rows of d_h fp32) exceed 200 KiB of shared memory";
        return false;
    }
    return true;
}

cudaError_t launch_topk(const Plan &P, const void *q, const void *k,
                        const int32_t *perm_q, const int32_t *perm_k,
                        float *sums, int32_t *cand, uint32_t *selmask,
                        DeviceStatus *status, cudaStream_t st) {
    const int T = P.N / P.b;
    dim3 gs(T, P.BH, 2);
    if (P.dtype == ELSAA_FP32)
        k_topk_sums<float><<<gs, P.d, 0, st>>>(
            (const float *)q, (const float *)k, perm_q, perm_k, P.N, P.d, P.b,
            sums, status);
    else
        k_topk_sums<__nv_bfloat16><<<gs, P.d, 0, st>>>(
            (const __nv_bfloat16 *)q, (const __nv_bfloat16 *)k, perm_q,
            perm_k, P.N, P.d, P.b, sums, status);
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return e;
    const size_t csm = (size_t)P.d * 4 + (size_t)T * 8;
    if (csm > 48 * 1024)
        cudaFuncSetAttribute(k_topk_cand,
                             cudaFuncAttributeMaxDynamicSharedMemorySize,
                             (int)csm);
    k_topk_cand<<<dim3(T, P.BH), kSelThreads, csm, st>>>(sums, P.d, P.tk_c,
                                                         cand);
    e = cudaGetLastError();
    if (e != cudaSuccess) return e;
    const size_t smem = select_smem(P);
    auto run = [&](auto kern, auto *qp, auto *kp) {
        cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             (int)smem);
        kern<<<dim3(T, P.BH), kSelThreads, smem, st>>>(
            qp, kp, perm_q, perm_k, cand, P.N, P.d, P.b, P.tk_c, P.tk_k,
            selmask, status);
        return cudaGetLastError();
    };
    const int M = P.tk_c * P.b / 32;
#define ELSAA_SEL_CASE(MM)                                                    \
    case MM:                                                                  \
        return P.dtype == ELSAA_FP32                                          \
                   ? run(k_topk_select<float, MM>, (const float *)q,          \
                         (const float *)k)                                    \
                   : run(k_topk_select<__nv_bfloat16, MM>,                    \
                         (const __nv_bfloat16 *)q,                            \
                         (const __nv_bfloat16 *)k);
    switch (M) {
        ELSAA_SEL_CASE(1)
        ELSAA_SEL_CASE(2)
        ELSAA_SEL_CASE(3)
        ELSAA_SEL_CASE(4)
        ELSAA_SEL_CASE(5)
        ELSAA_SEL_CASE(6)
        ELSAA_SEL_CASE(7)
        ELSAA_SEL_CASE(8)
        ELSAA_SEL_CASE(9)
        ELSAA_SEL_CASE(10)
        ELSAA_SEL_CASE(11)
        ELSAA_SEL_CASE(12)
        ELSAA_SEL_CASE(13)
        ELSAA_SEL_CASE(14)
        ELSAA_SEL_CASE(15)
        ELSAA_SEL_CASE(16)
        default: return cudaErrorInvalidValue;
    }
#undef ELSAA_SEL_CASE
}

cudaError_t launch_topk_export(const Plan &P, const int32_t *perm_q,
                               const int32_t *perm_k, const int32_t *cand,
                               const uint32_t *selmask, int32_t *out,
                               DeviceStatus *status, cudaStream_t st) {
    dim3 grid((P.N + kSelWarps - 1) / kSelWarps, P.BH);
    k_topk_export<<<grid, kSelThreads, 0, st>>>(perm_q, perm_k, cand, selmask,
                                                P.N, P.b, P.tk_c, P.tk_k, out,
                                                status);
    return cudaGetLastError();
}

}  // namespace elsaa
