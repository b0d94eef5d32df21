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
    // rows 16 at a time: the loads are issued together, the additions stay
    // in sorted order
    constexpr int kU = 16;
    float acc = 0.0f;
    for (int p0 = t * b; p0 < (t + 1) * b; p0 += kU) {
        float v[kU];
#pragma unroll
        for (int u = 0; u < kU; ++u) {
            int i = pm[p0 + u];
            if (i < 0 || i >= N) {
                if (e == 0) report(status, kDevPermRange, 20, bh, i);
                i = 0;
            }
            v[u] = to_f32<X>(x[(size_t)i * d + e]);
        }
#pragma unroll
        for (int u = 0; u < kU; ++u) acc = __fadd_rn(acc, v[u]);
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
        const float4 *kr = reinterpret_cast<const float4 *>(ksum +
                                                             (size_t)u * d);
        float acc = 0.0f;
        for (int e = 0; e < d; e += 16) {
            float4 kv[4];
#pragma unroll
            for (int x = 0; x < 4; ++x) kv[x] = kr[e / 4 + x];
#pragma unroll
            for (int x = 0; x < 4; ++x) {
                acc = fmaf(qs[e + 4 * x], kv[x].x, acc);
                acc = fmaf(qs[e + 4 * x + 1], kv[x].y, acc);
                acc = fmaf(qs[e + 4 * x + 2], kv[x].z, acc);
                acc = fmaf(qs[e + 4 * x + 3], kv[x].w, acc);
            }
        }
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

// Candidate-key staging element: bf16 inputs stay bf16 in shared memory
// (widened exactly when read), fp32 inputs stay fp32.
template <typename X>
struct SelStage;
template <>
struct SelStage<float> {
    using T = float;
    static constexpr int kPer16 = 4;  // values per 16-byte load
    __device__ static void widen(const uint4 &u, float *f) {
        f[0] = __uint_as_float(u.x);
        f[1] = __uint_as_float(u.y);
        f[2] = __uint_as_float(u.z);
        f[3] = __uint_as_float(u.w);
    }
};
template <>
struct SelStage<__nv_bfloat16> {
    using T = __nv_bfloat16;
    static constexpr int kPer16 = 8;
    __device__ static void widen(const uint4 &u, float *f) {
        const uint32_t w[4] = {u.x, u.y, u.z, u.w};
#pragma unroll
        for (int i = 0; i < 4; ++i) {
            f[2 * i] = __uint_as_float(w[i] << 16);
            f[2 * i + 1] = __uint_as_float(w[i] & 0xffff0000u);
        }
    }
};

// Rows of staged candidate keys: d + 16 bytes of padding keep 16-byte
// alignment and spread a quarter-warp's 16-byte loads over all banks.
template <typename X>
__host__ __device__ constexpr int sel_row_bytes(int d) {
    return d * (int)sizeof(X) + 16;
}

constexpr int kSelQB = 4;  // queries per warp sharing each key load

// 16-byte global -> shared copy that does not block the thread
// (cp.async.cg), and the wait for all of this thread's copies.
__device__ __forceinline__ void sel_cp16(void *dst, const void *src) {
    const uint32_t d =
        static_cast<uint32_t>(__cvta_generic_to_shared(dst));
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(d),
                 "l"(src)
                 : "memory");
}
__device__ __forceinline__ void sel_cp_wait() {
    asm volatile("cp.async.wait_all;" ::: "memory");
}

// Two fp32 lanes per instruction (fma.rn.f32x2): lane by lane d = a b + c,
// one rounding each, so each lane is an ordinary fmaf.
__device__ __forceinline__ unsigned long long sel_fma2(unsigned long long a,
                                                       unsigned long long b,
                                                       unsigned long long c) {
    unsigned long long r;
    asm("fma.rn.f32x2 %0, %1, %2, %3;" : "=l"(r) : "l"(a), "l"(b), "l"(c));
    return r;
}
__device__ __forceinline__ unsigned long long sel_pack(float lo, float hi) {
    unsigned long long r;
    asm("mov.b64 %0, {%1, %2};" : "=l"(r) : "f"(lo), "f"(hi));
    return r;
}
__device__ __forceinline__ float sel_lo(unsigned long long v) {
    return __uint_as_float((uint32_t)v);
}
__device__ __forceinline__ float sel_hi(unsigned long long v) {
    return __uint_as_float((uint32_t)(v >> 32));
}

// Grid (T, BH), kSelThreads threads, M = c b / 32 candidate words (<= 16).
// Dynamic shared memory: the candidate keys and the block's b queries (both
// in the input type, rows padded), the candidates' original indices. All
// rows are copied at once (indices first, then every 16-byte piece with
// cp.async). Each warp scores kSelQB queries at a time: every staged key
// value feeds two packed chains (queries 0|1 and 2|3), then the four radix
// selects run interleaved.
template <typename X, int M>
__global__ void __launch_bounds__(kSelThreads)
    k_topk_select(const X *__restrict__ qx, const X *__restrict__ kx,
                  const int32_t *__restrict__ perm_q,
                  const int32_t *__restrict__ perm_k,
                  const int32_t *__restrict__ cand, int N, int d, int b,
                  int c, int k, uint32_t *__restrict__ selmask,
                  DeviceStatus *status) {
    using S = SelStage<X>;
    extern __shared__ __align__(16) unsigned char sel_smem[];
    const int t = blockIdx.x, bh = blockIdx.y, T = gridDim.x;
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int nc = 32 * M, rb = sel_row_bytes<X>(d);
    unsigned char *kc = sel_smem;                                 // [nc][rb]
    unsigned char *qs = kc + (size_t)nc * rb;                     // [b][rb]
    int *cidx = reinterpret_cast<int *>(qs + (size_t)b * rb);     // [nc]
    int *qidx = cidx + nc;                                        // [b]
    const X *qh = qx + (size_t)bh * N * d;
    const X *kh = kx + (size_t)bh * N * d;
    const int32_t *pq = perm_q + (size_t)bh * N;
    const int32_t *pk = perm_k + (size_t)bh * N;
    const int32_t *cb = cand + ((size_t)bh * T + t) * c;
    // the c b candidate keys (candidate r = key r % b of block r / b) and
    // the block's queries: original indices first, then the rows
    for (int r = tid; r < nc; r += kSelThreads) {
        int u = cb[r / b];
        if (u < 0 || u >= T) u = t;
        int j = pk[u * b + r % b];
        if (j < 0 || j >= N) {
            report(status, kDevPermRange, 21, bh, j);
            j = 0;
        }
        cidx[r] = j;
    }
    for (int r = tid; r < b; r += kSelThreads) {
        int i = pq[t * b + r];
        if (i < 0 || i >= N) {
            report(status, kDevPermRange, 22, bh, i);
            i = 0;
        }
        qidx[r] = i;
    }
    __syncthreads();
    const int cpr = d * (int)sizeof(X) / 16;  // 16-byte chunks per row
    for (int x = tid; x < nc * cpr; x += kSelThreads) {
        const int r = x / cpr, ch = x - r * cpr;
        sel_cp16(kc + (size_t)r * rb + 16 * ch,
                 reinterpret_cast<const unsigned char *>(
                     kh + (size_t)cidx[r] * d) + 16 * ch);
    }
    for (int x = tid; x < b * cpr; x += kSelThreads) {
        const int r = x / cpr, ch = x - r * cpr;
        sel_cp16(qs + (size_t)r * rb + 16 * ch,
                 reinterpret_cast<const unsigned char *>(
                     qh + (size_t)qidx[r] * d) + 16 * ch);
    }
    sel_cp_wait();
    __syncthreads();
    int cj[M];  // original index of each of this lane's candidates
#pragma unroll
    for (int m = 0; m < M; ++m) cj[m] = cidx[lane + 32 * m];
    const int W = M;  // mask words per query
    for (int q0 = warp * kSelQB; q0 < b; q0 += kSelWarps * kSelQB) {
        const int nq = min(kSelQB, b - q0);
        // query rows of this group (rows past the block repeat row q0)
        const unsigned char *qr[kSelQB];
#pragma unroll
        for (int qq = 0; qq < kSelQB; ++qq)
            qr[qq] = qs + (size_t)(q0 + (qq < nq ? qq : 0)) * rb;
        // canonical chains: query qq, candidate lane + 32 m, e = 0 .. d - 1
        // in order (each lane of a packed fma rounds once, from +0.0f)
        unsigned long long acc01[M], acc23[M];
#pragma unroll
        for (int m = 0; m < M; ++m) acc01[m] = acc23[m] = 0ull;
        for (int e0 = 0; e0 < d; e0 += S::kPer16) {
            unsigned long long q01[S::kPer16], q23[S::kPer16];
            {
                float qv[kSelQB][S::kPer16];
#pragma unroll
                for (int qq = 0; qq < kSelQB; ++qq)
                    S::widen(*reinterpret_cast<const uint4 *>(
                                 qr[qq] + e0 * (int)sizeof(X)),
                             qv[qq]);
#pragma unroll
                for (int x = 0; x < S::kPer16; ++x) {
                    q01[x] = sel_pack(qv[0][x], qv[1][x]);
                    q23[x] = sel_pack(qv[2][x], qv[3][x]);
                }
            }
#pragma unroll
            for (int m = 0; m < M; ++m) {
                const uint4 u = *reinterpret_cast<const uint4 *>(
                    kc + (size_t)(lane + 32 * m) * rb +
                    e0 * (int)sizeof(X));
                float kv[S::kPer16];
                S::widen(u, kv);
#pragma unroll
                for (int x = 0; x < S::kPer16; ++x) {
                    const unsigned long long kk = sel_pack(kv[x], kv[x]);
                    acc01[m] = sel_fma2(q01[x], kk, acc01[m]);
                    acc23[m] = sel_fma2(q23[x], kk, acc23[m]);
                }
            }
        }
        uint32_t key[kSelQB][M];
#pragma unroll
        for (int m = 0; m < M; ++m) {
            key[0][m] = ordered_key(sel_lo(acc01[m]));
            key[1][m] = ordered_key(sel_hi(acc01[m]));
            key[2][m] = ordered_key(sel_lo(acc23[m]));
            key[3][m] = ordered_key(sel_hi(acc23[m]));
        }
        // the k-th largest key of each query: the largest value T with at
        // least k keys >= T, built MSB first (a bit stays set when enough
        // keys reach it); the four searches run together, two counts packed
        // per warp reduction
        uint32_t pre[kSelQB] = {0u, 0u, 0u, 0u};
        for (int bit = 31; bit >= 0; --bit) {
            const uint32_t bm = 1u << bit;
            int cnt[kSelQB];
#pragma unroll
            for (int qq = 0; qq < kSelQB; ++qq) {
                const uint32_t want = pre[qq] | bm;
                int n = 0;
#pragma unroll
                for (int m = 0; m < M; ++m) n += key[qq][m] >= want;
                cnt[qq] = n;
            }
            const int c01 = __reduce_add_sync(0xffffffffu,
                                              cnt[0] | (cnt[1] << 16));
            const int c23 = __reduce_add_sync(0xffffffffu,
                                              cnt[2] | (cnt[3] << 16));
            cnt[0] = c01 & 0xffff;
            cnt[1] = c01 >> 16;
            cnt[2] = c23 & 0xffff;
            cnt[3] = c23 >> 16;
#pragma unroll
            for (int qq = 0; qq < kSelQB; ++qq)
                if (cnt[qq] >= k) pre[qq] |= bm;
        }
        // keys strictly above each threshold
        int above[kSelQB];
        {
            int cnt[kSelQB];
#pragma unroll
            for (int qq = 0; qq < kSelQB; ++qq) {
                int n = 0;
#pragma unroll
                for (int m = 0; m < M; ++m) n += key[qq][m] > pre[qq];
                cnt[qq] = n;
            }
            const int c01 = __reduce_add_sync(0xffffffffu,
                                              cnt[0] | (cnt[1] << 16));
            const int c23 = __reduce_add_sync(0xffffffffu,
                                              cnt[2] | (cnt[3] << 16));
            above[0] = c01 & 0xffff;
            above[1] = c01 >> 16;
            above[2] = c23 & 0xffff;
            above[3] = c23 >> 16;
        }
        for (int qq = 0; qq < nq; ++qq) {
            const int p = t * b + q0 + qq;
            // keys equal to the threshold: the need lowest original indices
            const int need = k - above[qq];
            int ties = 0;
#pragma unroll
            for (int m = 0; m < M; ++m) ties += key[qq][m] == pre[qq];
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
                        cnt += key[qq][m] == pre[qq] &&
                               ((uint32_t)cj[m] & mk) == jp;
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
                const bool sl = key[qq][m] > pre[qq] ||
                                (key[qq][m] == pre[qq] && cj[m] <= jmax);
                const uint32_t word = __ballot_sync(0xffffffffu, sl);
                if (lane == m) out[m] = word;
            }
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
    const int rb = P.dtype == ELSAA_FP32 ? sel_row_bytes<float>(P.d)
                                         : sel_row_bytes<__nv_bfloat16>(P.d);
    return (size_t)(nc + P.b) * rb + (size_t)(nc + P.b) * 4;
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
               "block_size rows of d_h values) exceed 200 KiB of shared "
               "memory";
        return false;
    }
    return true;
}

cudaError_t launch_topk(int stage, const Plan &P, const void *q,
                        const void *k, const int32_t *perm_q,
                        const int32_t *perm_k, float *sums, int32_t *cand,
                        uint32_t *selmask, DeviceStatus *status,
                        cudaStream_t st) {
    const int T = P.N / P.b;
    if (stage == 0) {
    dim3 gs(T, P.BH, 2);
    if (P.dtype == ELSAA_FP32)
        k_topk_sums<float><<<gs, P.d, 0, st>>>(
            (const float *)q, (const float *)k, perm_q, perm_k, P.N, P.d, P.b,
            sums, status);
    else
        k_topk_sums<__nv_bfloat16><<<gs, P.d, 0, st>>>(
            (const __nv_bfloat16 *)q, (const __nv_bfloat16 *)k, perm_q,
            perm_k, P.N, P.d, P.b, sums, status);
        return cudaGetLastError();
    }
    if (stage == 1) {
        const size_t csm = (size_t)P.d * 4 + (size_t)T * 8;
        if (csm > 48 * 1024)
            cudaFuncSetAttribute(k_topk_cand,
                                 cudaFuncAttributeMaxDynamicSharedMemorySize,
                                 (int)csm);
        k_topk_cand<<<dim3(T, P.BH), kSelThreads, csm, st>>>(sums, P.d,
                                                             P.tk_c, cand);
        return cudaGetLastError();
    }
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
