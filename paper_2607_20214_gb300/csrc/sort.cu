// sortLSH selection: angular sort hash, stable counting sort, block order.
//
// Algorithm "sortLSH Sparse Exact Attention Branch", steps Hash and Sort:
// every query and key gets an n_s-bit angular hash (bit p = sign of the
// projection on plane p, Section 3.2 / Appendix F), the codes are ordered
// by their rank in the reflected Gray sequence (sorted Hamming LSH,
// Section 3), and P_Q, P_K stably sort the keys (equal keys keep increasing
// original index). Consecutive runs of b sorted positions form the blocks.
//
// Three launches, all integer-exact after the hash:
//   sort_hash    one CTA per 128-token tile of (head, Q|K): hash, tile
//                histogram, rank of each token among equal keys of its tile.
//   sort_scan    one CTA per (head, Q|K): exclusive scan of the tile
//                histograms in (bin, tile) order -> start offset of every
//                (tile, bin) run in the sorted order.
//   sort_scatter one CTA per tile: pos = offset[tile][key] + local rank,
//                perm[pos] = token.
#include "device_common.cuh"

namespace elsaa {

namespace {

template <typename T>
__global__ void __launch_bounds__(kHashTile)
    k_sort_hash(const T *__restrict__ q, const T *__restrict__ k,
                const float *__restrict__ w_sort, int N, int d, int H,
                int n_s, int bins, int gray, int tiles,
                uint32_t *__restrict__ keyrank, int *__restrict__ hist) {
    extern __shared__ float smem[];
    const int tile = blockIdx.x, bh = blockIdx.y, which = blockIdx.z;
    const int BH = gridDim.y;
    const int tid = threadIdx.x;
    const int h = bh % H;
    const int ds = d + 1;  // padded row stride: conflict-free column walks
    float *xs = smem;                      // [kHashTile][d + 1]
    float *ws = xs + kHashTile * ds;       // [n_s][d]
    int *keys = (int *)(ws + n_s * d);     // [kHashTile]
    int *hs = keys + kHashTile;            // [bins]

    const T *x = (which ? k : q) + (size_t)bh * N * d;
    const int n0 = tile * kHashTile;
    for (int i = tid; i < kHashTile * d; i += kHashTile) {
        int row = i / d, col = i - row * d;
        int n = n0 + row;
        xs[row * ds + col] = n < N ? to_f32<T>(x[(size_t)n * d + col]) : 0.f;
    }
    for (int i = tid; i < n_s * d; i += kHashTile)
        ws[i] = w_sort[(size_t)h * n_s * d + i];
    for (int i = tid; i < bins; i += kHashTile) hs[i] = 0;
    __syncthreads();

    const int n = n0 + tid;
    int key = -1;
    if (n < N) {
        uint32_t code = 0;
        const float *xr = xs + tid * ds;
        for (int p = 0; p < n_s; ++p) {
            // canonical projection: sequential fp32 FMA chain, i = 0..d-1
            float acc = 0.0f;
            const float *wp = ws + p * d;
            for (int e = 0; e < d; ++e) acc = __fmaf_rn(wp[e], xr[e], acc);
            code |= (acc > 0.0f ? 1u : 0u) << p;
        }
        key = (int)(gray ? gray_rank(code) : code);
    }
    keys[tid] = key;
    __syncthreads();
    if (n < N) {
        int rank = 0;
        for (int j = 0; j < tid; ++j) rank += keys[j] == key;
        atomicAdd(&hs[key], 1);
        keyrank[((size_t)which * BH + bh) * N + n] =
            (uint32_t)key | ((uint32_t)rank << 16);
    }
    __syncthreads();
    int *hout = hist + (((size_t)which * BH + bh) * tiles + tile) * bins;
    for (int i = tid; i < bins; i += kHashTile) hout[i] = hs[i];
}

constexpr int kScanThreads = 1024;

__global__ void __launch_bounds__(kScanThreads)
    k_sort_scan(int *__restrict__ hist, int tiles, int bins) {
    __shared__ int warp_tot[32];
    const int tid = threadIdx.x;
    int *hst = hist + (size_t)blockIdx.x * tiles * bins;  // [tiles][bins]
    const long E = (long)tiles * bins;                    // bin-major order
    const long per = (E + kScanThreads - 1) / kScanThreads;
    const long e0 = tid * per;
    const long e1 = e0 + per < E ? e0 + per : E;
    int sum = 0;
    for (long e = e0; e < e1; ++e) {
        int bin = (int)(e / tiles), t = (int)(e - (long)bin * tiles);
        sum += hst[(size_t)t * bins + bin];
    }
    // block exclusive scan of per-thread sums
    const int lane = tid & 31, wid = tid >> 5;
    int incl = sum;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        int y = __shfl_up_sync(0xffffffffu, incl, o);
        if (lane >= o) incl += y;
    }
    if (lane == 31) warp_tot[wid] = incl;
    __syncthreads();
    if (wid == 0) {
        int w = warp_tot[lane];
        int wi = w;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            int y = __shfl_up_sync(0xffffffffu, wi, o);
            if (lane >= o) wi += y;
        }
        warp_tot[lane] = wi - w;  // exclusive warp offsets
    }
    __syncthreads();
    int run = warp_tot[wid] + incl - sum;
    for (long e = e0; e < e1; ++e) {
        int bin = (int)(e / tiles), t = (int)(e - (long)bin * tiles);
        int c = hst[(size_t)t * bins + bin];
        hst[(size_t)t * bins + bin] = run;
        run += c;
    }
}

__global__ void __launch_bounds__(kHashTile)
    k_sort_scatter(const uint32_t *__restrict__ keyrank,
                   const int *__restrict__ hist, int N, int tiles, int bins,
                   int32_t *__restrict__ perm_q, int32_t *__restrict__ perm_k,
                   DeviceStatus *status) {
    const int tile = blockIdx.x, bh = blockIdx.y, which = blockIdx.z;
    const int BH = gridDim.y;
    const int n = tile * kHashTile + threadIdx.x;
    if (n >= N) return;
    uint32_t kr = keyrank[((size_t)which * BH + bh) * N + n];
    int key = (int)(kr & 0xffffu), rank = (int)(kr >> 16);
    int pos = hist[(((size_t)which * BH + bh) * tiles + tile) * bins + key] +
              rank;
    if (pos < 0 || pos >= N) {
        report(status, kDevSortRange, 0, bh, pos);
        return;
    }
    int32_t *perm = (which ? perm_k : perm_q) + (size_t)bh * N;
    perm[pos] = n;
}

}  // namespace

cudaError_t launch_sort_hash(const Plan &P, const void *q, const void *k,
                             const float *w_sort, uint32_t *keyrank,
                             int *hist, cudaStream_t st) {
    dim3 grid(P.tiles, P.BH, 2);
    size_t smem = sizeof(float) * ((size_t)kHashTile * (P.d + 1) +
                                   (size_t)P.n_s * P.d) +
                  sizeof(int) * (kHashTile + P.bins);
    if (P.dtype == ELSAA_FP32) {
        auto kern = k_sort_hash<float>;
        cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             (int)smem);
        kern<<<grid, kHashTile, smem, st>>>(
            (const float *)q, (const float *)k, w_sort, P.N, P.d, P.H, P.n_s,
            P.bins, P.gray, P.tiles, keyrank, hist);
    } else {
        auto kern = k_sort_hash<__nv_bfloat16>;
        cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             (int)smem);
        kern<<<grid, kHashTile, smem, st>>>(
            (const __nv_bfloat16 *)q, (const __nv_bfloat16 *)k, w_sort, P.N,
            P.d, P.H, P.n_s, P.bins, P.gray, P.tiles, keyrank, hist);
    }
    return cudaGetLastError();
}

cudaError_t launch_sort_scan(const Plan &P, int *hist, cudaStream_t st) {
    k_sort_scan<<<2 * P.BH, kScanThreads, 0, st>>>(hist, P.tiles, P.bins);
    return cudaGetLastError();
}

cudaError_t launch_sort_scatter(const Plan &P, const uint32_t *keyrank,
                                const int *hist, int32_t *perm_q,
                                int32_t *perm_k, DeviceStatus *status,
                                cudaStream_t st) {
    dim3 grid(P.tiles, P.BH, 2);
    k_sort_scatter<<<grid, kHashTile, 0, st>>>(keyrank, hist, P.N, P.tiles,
                                               P.bins, perm_q, perm_k, status);
    return cudaGetLastError();
}

}  // namespace elsaa
