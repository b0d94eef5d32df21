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
//   sort_hash    one CTA per two 128-token tiles of (head, Q|K): hash,
//                tile histograms, rank of each token among equal keys of
//                its tile.
//   sort_scan    one CTA per (head, Q|K): exclusive scan of the tile
//                histograms stored bin-major ([bin][tile]) -> start offset
//                of every (tile, bin) run in the sorted order.
//   sort_scatter one CTA per tile: pos = offset[tile][key] + local rank,
//                perm[pos] = token.
#include "device_common.cuh"
#include "tc_common.cuh"

namespace elsaa {

namespace {

template <typename T>
__device__ __forceinline__ void unpack8(const uint4 &u, float *x);
template <>
__device__ __forceinline__ void unpack8<__nv_bfloat16>(const uint4 &u,
                                                       float *x) {
    const uint32_t w[4] = {u.x, u.y, u.z, u.w};
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        x[2 * i] = __uint_as_float(w[i] << 16);
        x[2 * i + 1] = __uint_as_float(w[i] & 0xffff0000u);
    }
}

template <>
__device__ __forceinline__ void unpack8<float>(const uint4 &u, float *x) {
    x[0] = __uint_as_float(u.x);
    x[1] = __uint_as_float(u.y);
    x[2] = __uint_as_float(u.z);
    x[3] = __uint_as_float(u.w);
}

// Two fp32 FMAs in one instruction: lanes (lo, hi) of d = a * b + c, each an
// IEEE round-to-nearest fused multiply-add (bit-identical to fmaf).
__device__ __forceinline__ unsigned long long fma2(unsigned long long a,
                                                   unsigned long long b,
                                                   unsigned long long c) {
    unsigned long long d;
    asm("fma.rn.f32x2 %0, %1, %2, %3;" : "=l"(d) : "l"(a), "l"(b), "l"(c));
    return d;
}
__device__ __forceinline__ unsigned long long pair2(float lo, float hi) {
    return ((unsigned long long)__float_as_uint(hi) << 32) |
           __float_as_uint(lo);
}

// One CTA hashes two 128-token tiles (A = 2 * blockIdx.x, B = A + 1) of one
// (head, Q|K). The tiles are staged in shared memory with cp.async (16-byte
// chunks of each row XOR-swizzled by the row index, so a warp reading one
// chunk of 32 rows is conflict-free). Thread t evaluates the NS projections
// of row t of both tiles with packed fma.rn.f32x2 (lane lo: tile A, lane
// hi: tile B); every chain keeps the canonical sequential order
// i = 0..d-1. Ranks among equal keys of a tile come from warp match masks
// plus per-warp counts.
template <typename T, int NS>
__global__ void __launch_bounds__(kHashTile)
    k_sort_hash(const T *__restrict__ q, const T *__restrict__ k,
                const float *__restrict__ w_sort, int N, int d, int H,
                int bins, int gray, int tiles, uint32_t *__restrict__ keyrank,
                int *__restrict__ hist) {
    extern __shared__ __align__(16) unsigned char smem[];
    const int tile0 = 2 * blockIdx.x, bh = blockIdx.y, which = blockIdx.z;
    const int BH = gridDim.y;
    const int tid = threadIdx.x, lane = tid & 31, wid = tid >> 5;
    const int h = bh % H;
    constexpr int kEl = 16 / sizeof(T);          // elements per 16-byte chunk
    const int cpr = d / kEl;                     // chunks per row
    const int swz = cpr >= 8 ? 7 : cpr - 1;      // swizzle mask
    uint4 *xs = reinterpret_cast<uint4 *>(smem);  // [2][128][cpr]
    float *ws = reinterpret_cast<float *>(xs + 2 * kHashTile * cpr);  // [NS][d]
    int *cnt = reinterpret_cast<int *>(ws + NS * d);  // [2][4 warps][bins]

    const T *x = (which ? k : q) + (size_t)bh * N * d;
    const uint32_t xs_s = static_cast<uint32_t>(__cvta_generic_to_shared(xs));
    for (int tt = 0; tt < 2; ++tt) {
        const int n0 = (tile0 + tt) * kHashTile;
        const int valid_rows = max(0, min(kHashTile, N - n0));
        const uint4 *src = reinterpret_cast<const uint4 *>(x + (size_t)n0 * d);
        for (int i = tid; i < kHashTile * cpr; i += kHashTile) {
            int row = i / cpr, c = i - row * cpr;
            int slot = (tt * kHashTile + row) * cpr + (c ^ (row & swz));
            if (row < valid_rows)
                asm volatile(
                    "cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(
                        xs_s + 16u * slot),
                    "l"(src + (size_t)row * cpr + c)
                    : "memory");
            else
                xs[slot] = make_uint4(0u, 0u, 0u, 0u);
        }
    }
    asm volatile("cp.async.commit_group;" ::: "memory");
    for (int i = tid; i < NS * d; i += kHashTile)
        ws[i] = w_sort[(size_t)h * NS * d + i];
    for (int i = tid; i < 8 * bins; i += kHashTile) cnt[i] = 0;
    asm volatile("cp.async.wait_all;" ::: "memory");
    __syncthreads();

    unsigned long long acc[NS > 0 ? NS : 1];
#pragma unroll
    for (int p = 0; p < NS; ++p) acc[p] = 0ull;
    const uint4 *xa = xs + tid * cpr;
    const uint4 *xb = xs + (kHashTile + tid) * cpr;
    const float4 *ws4 = reinterpret_cast<const float4 *>(ws);
    for (int c = 0; c < cpr; ++c) {
        float va[kEl], vb[kEl];
        unpack8<T>(xa[c ^ (tid & swz)], va);
        unpack8<T>(xb[c ^ (tid & swz)], vb);
        const int e0 = c * kEl;
#pragma unroll
        for (int j = 0; j < kEl / 4; ++j) {
            float wv[NS > 0 ? NS : 1][4];
#pragma unroll
            for (int p = 0; p < NS; ++p) {
                float4 w4 = ws4[(p * d + e0) / 4 + j];  // same for all lanes
                wv[p][0] = w4.x;
                wv[p][1] = w4.y;
                wv[p][2] = w4.z;
                wv[p][3] = w4.w;
            }
#pragma unroll
            for (int e = 0; e < 4; ++e) {
                const unsigned long long xp = pair2(va[4 * j + e], vb[4 * j + e]);
#pragma unroll
                for (int p = 0; p < NS; ++p)
                    acc[p] = fma2(pair2(wv[p][e], wv[p][e]), xp, acc[p]);
            }
        }
    }
    int *hout = hist + ((size_t)which * BH + bh) * tiles * bins;
#pragma unroll
    for (int tt = 0; tt < 2; ++tt) {
        const int tile = tile0 + tt;
        const int n = tile * kHashTile + tid;
        uint32_t code = 0;
#pragma unroll
        for (int p = 0; p < NS; ++p) {
            const float pr = __uint_as_float(
                (uint32_t)(tt ? (acc[p] >> 32) : (acc[p] & 0xffffffffull)));
            code |= (pr > 0.0f ? 1u : 0u) << p;
        }
        const int key = (int)(gray ? gray_rank(code) : code);
        const bool in = n < N && tile < tiles;
        const unsigned act = __ballot_sync(0xffffffffu, in);
        unsigned peers = __match_any_sync(0xffffffffu, in ? key : -1) & act;
        const int rank_w = __popc(peers & ((1u << lane) - 1u));
        int *cw = cnt + tt * 4 * bins;
        if (in && rank_w == 0) cw[wid * bins + key] = __popc(peers);
        __syncthreads();
        if (in) {
            int rank = rank_w;
            for (int w = 0; w < wid; ++w) rank += cw[w * bins + key];
            keyrank[((size_t)which * BH + bh) * N + n] =
                (uint32_t)key | ((uint32_t)rank << 16);
        }
        // tile histogram, stored bin-major ([bins][tiles]) so that the scan
        // walks one contiguous array
        if (tile < tiles)
            for (int i = tid; i < bins; i += kHashTile)
                hout[(size_t)i * tiles + tile] = cw[i] + cw[bins + i] +
                                                 cw[2 * bins + i] +
                                                 cw[3 * bins + i];
    }
}

// k_sort_hash_tma: warps 0-3 hash, warp 4 streams the inputs with TMA.
// A work item is four consecutive 128-token tiles (512 rows) of one
// (head, Q|K); a job is one 32-column panel of an item (64 bytes per row,
// 64-byte swizzle: 16-byte chunk c of row r sits at chunk c ^ ((r >> 1) & 3)),
// loaded as two 256-row boxes into one stage of a three-stage ring. Two
// CTAs share an SM.
constexpr int kHashStages = 3;
constexpr int kHashItemTiles = 4;
constexpr int kHashRows = kHashItemTiles * kHashTile;
constexpr int kHashBoxRows = 256;
constexpr int kHashCols = 32;
constexpr uint32_t kHashStageBytes = kHashRows * kHashCols * 2;
constexpr int kHashThreads = kHashTile + 32;

// bf16 inputs with d in {64, 128}: the same hash, ranks and histograms as
// k_sort_hash, from persistent CTAs whose producer warp keeps the next
// panels in flight while the hashing warps work. CTA c owns a contiguous
// range of items (items of one head are adjacent, so the planes are
// reloaded only when the head changes). Hashing thread t evaluates rows
// t, 128 + t, 256 + t and 384 + t of the item as two packed chains
// (fma.rn.f32x2 lanes: tiles 0|1 and tiles 2|3); the planes sit in shared
// memory as duplicated pairs (w, w), so one 16-byte load feeds four packed
// FMAs. Every chain keeps the canonical sequential order i = 0..d-1.
template <int NS>
__global__ void __launch_bounds__(kHashThreads, 2)
    k_sort_hash_tma(const __grid_constant__ CUtensorMap tmQ,
                    const __grid_constant__ CUtensorMap tmK,
                    const float *__restrict__ w_sort, int N, int d, int H,
                    int BH, int bins, int gray, int tiles, int quads,
                    int items, int per_cta, uint32_t *__restrict__ keyrank,
                    int *__restrict__ hist, DeviceStatus *status) {
    using namespace tc;
    extern __shared__ unsigned char smem_raw[];
    __shared__ uint64_t full[kHashStages], empty[kHashStages];
    __shared__ int abort_flag;
    // 512-byte aligned start, the period of the 64-byte swizzle (pointer
    // arithmetic on the shared array keeps every access an ld.shared)
    unsigned char *smem =
        smem_raw + ((512u - (smem_u32(smem_raw) & 511u)) & 511u);
    const uint32_t stage0 = smem_u32(smem);
    float2 *ws2 = reinterpret_cast<float2 *>(smem + kHashStages *
                                             kHashStageBytes);  // [NS][d]
    int *cnt = reinterpret_cast<int *>(ws2 + NS * d);  // [4 tiles][4 w][bins]
    const int tid = threadIdx.x, lane = tid & 31, wid = tid >> 5;
    const int P = d / kHashCols;  // panels per row
    const int i0 = blockIdx.x * per_cta;
    const int i1 = min(items, i0 + per_cta);
    if (i0 >= i1) return;
    const int njobs = (i1 - i0) * P;

    if (tid == 0) {
        for (int s = 0; s < kHashStages; ++s) {
            mbar_init(&full[s], 1);
            mbar_init(&empty[s], kHashTile / 32);
        }
        abort_flag = 0;
        fence_mbar_init();
    }
    __syncthreads();

    if (wid == kHashTile / 32) {
        // ---- producer warp: job j = panel (j mod P) of item i0 + j / P
        if (lane == 0) {
            int it = i0, pnl = 0;
            int issued = 0;
            for (int j = 0; j < njobs; ++j) {
                const int s = j % kHashStages;
                if (j >= kHashStages &&
                    !mbar_wait_or_abort(&empty[s],
                                        ((j / kHashStages) - 1) & 1,
                                        &abort_flag, status, 0x5002))
                    break;
                const int bw = it / quads, quad = it - bw * quads;
                const int which = bw & 1, bh = bw >> 1;
                const int row = bh * N + quad * kHashRows;
                const uint32_t dst = stage0 + s * kHashStageBytes;
                const CUtensorMap *map = which ? &tmK : &tmQ;
                mbar_expect_tx(&full[s], kHashStageBytes);
                tma_load_2d(dst, map, pnl * kHashCols, row, &full[s]);
                tma_load_2d(dst + kHashStageBytes / 2, map, pnl * kHashCols,
                            row + kHashBoxRows, &full[s]);
                ++issued;
                if (++pnl == P) {
                    pnl = 0;
                    ++it;
                }
            }
            // never leave with copies in flight into this CTA's stages:
            // wait (bounded) for the last job issued into every stage
            for (int s = 0; s < kHashStages; ++s) {
                int last = issued - 1 - ((issued - 1 - s) % kHashStages +
                                         kHashStages) % kHashStages;
                if (last >= 0 && last < issued)
                    mbar_wait(&full[s], (last / kHashStages) & 1, status,
                              0x5003);
            }
        }
        return;
    }

    // ---- hashing warps
    int cur_h = -1;
    int j = 0;
    bool ok = true;
    for (int it = i0; it < i1 && ok; ++it) {
        const int bw = it / quads, quad = it - bw * quads;
        const int which = bw & 1, bh = bw >> 1;
        const int h = bh % H;
        if (h != cur_h) {  // uniform: planes of the new head, as (w, w)
            for (int i = tid; i < NS * d; i += kHashTile) {
                const float w = w_sort[(size_t)h * NS * d + i];
                ws2[i] = make_float2(w, w);
            }
            cur_h = h;
        }
        for (int i = tid; i < 4 * 4 * bins; i += kHashTile) cnt[i] = 0;
        named_sync(1, kHashTile);

        unsigned long long acc0[NS > 0 ? NS : 1], acc1[NS > 0 ? NS : 1];
#pragma unroll
        for (int p = 0; p < NS; ++p) acc0[p] = acc1[p] = 0ull;
        const int sw = (tid >> 1) & 3;  // same for rows 128k + t
        for (int pnl = 0; pnl < P; ++pnl, ++j) {
            const int s = j % kHashStages;
            ok = mbar_wait_or_abort(&full[s], (j / kHashStages) & 1,
                                    &abort_flag, status, 0x5001);
            if (!ok) break;
            const unsigned char *st = smem + s * kHashStageBytes;
            const uint4 *x0p = reinterpret_cast<const uint4 *>(
                st + tid * (kHashCols * 2));
            constexpr int kTileU4 = kHashTile * kHashCols * 2 / 16;
            // (w_i, w_i) and (w_i+1, w_i+1) as two packed operands
            const ulonglong2 *w4 = reinterpret_cast<const ulonglong2 *>(ws2);
#pragma unroll
            for (int c = 0; c < kHashCols / 8; ++c) {
                float v0[8], v1[8], v2[8], v3[8];
                unpack8<__nv_bfloat16>(x0p[(c ^ sw)], v0);
                unpack8<__nv_bfloat16>(x0p[kTileU4 + (c ^ sw)], v1);
                unpack8<__nv_bfloat16>(x0p[2 * kTileU4 + (c ^ sw)], v2);
                unpack8<__nv_bfloat16>(x0p[3 * kTileU4 + (c ^ sw)], v3);
                const int e0 = pnl * kHashCols + c * 8;
#pragma unroll
                for (int e2 = 0; e2 < 4; ++e2) {
                    const unsigned long long xa0 =
                        pair2(v0[2 * e2], v1[2 * e2]);
                    const unsigned long long xa1 =
                        pair2(v0[2 * e2 + 1], v1[2 * e2 + 1]);
                    const unsigned long long xb0 =
                        pair2(v2[2 * e2], v3[2 * e2]);
                    const unsigned long long xb1 =
                        pair2(v2[2 * e2 + 1], v3[2 * e2 + 1]);
#pragma unroll
                    for (int p = 0; p < NS; ++p) {
                        // same address in every lane (broadcast)
                        const ulonglong2 wq = w4[(p * d + e0) / 2 + e2];
                        acc0[p] = fma2(wq.x, xa0, acc0[p]);
                        acc1[p] = fma2(wq.x, xb0, acc1[p]);
                        acc0[p] = fma2(wq.y, xa1, acc0[p]);
                        acc1[p] = fma2(wq.y, xb1, acc1[p]);
                    }
                }
            }
            // this warp is done reading stage s
            __syncwarp();
            if (lane == 0) mbar_arrive(&empty[s]);
        }
        ok = named_sync_and(1, kHashTile, ok);
        if (!ok) break;

        int *hout = hist + ((size_t)which * BH + bh) * tiles * bins;
#pragma unroll
        for (int tt = 0; tt < kHashItemTiles; ++tt) {
            const int tile = kHashItemTiles * quad + tt;
            const int n = tile * kHashTile + tid;
            const unsigned long long *acc = tt < 2 ? acc0 : acc1;
            uint32_t code = 0;
#pragma unroll
            for (int p = 0; p < NS; ++p) {
                const float pr = __uint_as_float((uint32_t)(
                    (tt & 1) ? (acc[p] >> 32) : (acc[p] & 0xffffffffull)));
                code |= (pr > 0.0f ? 1u : 0u) << p;
            }
            const int key = (int)(gray ? gray_rank(code) : code);
            const bool in = n < N && tile < tiles;
            const unsigned act = __ballot_sync(0xffffffffu, in);
            unsigned peers =
                __match_any_sync(0xffffffffu, in ? key : -1) & act;
            const int rank_w = __popc(peers & ((1u << lane) - 1u));
            int *cw = cnt + tt * 4 * bins;
            if (in && rank_w == 0) cw[wid * bins + key] = __popc(peers);
            named_sync(1, kHashTile);
            if (in) {
                int rank = rank_w;
                for (int w = 0; w < wid; ++w) rank += cw[w * bins + key];
                keyrank[((size_t)which * BH + bh) * N + n] =
                    (uint32_t)key | ((uint32_t)rank << 16);
            }
            if (tile < tiles)
                for (int i = tid; i < bins; i += kHashTile)
                    hout[(size_t)i * tiles + tile] =
                        cw[i] + cw[bins + i] + cw[2 * bins + i] +
                        cw[3 * bins + i];
        }
        named_sync(1, kHashTile);  // counts and planes may be overwritten
    }
}

constexpr int kScanThreads = 1024;

// Exclusive scan of the [bins][tiles] histogram of one (head, Q|K) in place:
// entry (bin, tile) becomes the sorted position where that tile's run of
// `bin` keys starts. Each thread owns one contiguous segment.
__global__ void __launch_bounds__(kScanThreads)
    k_sort_scan(int *__restrict__ hist, int tiles, int bins) {
    __shared__ int warp_tot[32];
    const int tid = threadIdx.x;
    int *hst = hist + (size_t)blockIdx.x * tiles * bins;
    const int E = tiles * bins;
    const int per = (E + kScanThreads - 1) / kScanThreads;
    const int e0 = min(E, tid * per);
    const int e1 = min(E, e0 + per);
    int sum = 0;
    // 16-byte vector path when every segment start and end is 16-byte
    // aligned (E and per multiples of 4; the workspace is 256-byte aligned)
    const bool vec = ((per | E) & 3) == 0;
    if (vec) {
        for (int e = e0; e < e1; e += 4) {
            int4 v = *reinterpret_cast<const int4 *>(hst + e);
            sum += v.x + v.y + v.z + v.w;
        }
    } else {
        for (int e = e0; e < e1; ++e) sum += hst[e];
    }
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
    if (vec) {
        for (int e = e0; e < e1; e += 4) {
            int4 v = *reinterpret_cast<const int4 *>(hst + e);
            int4 o;
            o.x = run;
            o.y = o.x + v.x;
            o.z = o.y + v.y;
            o.w = o.z + v.z;
            run = o.w + v.w;
            *reinterpret_cast<int4 *>(hst + e) = o;
        }
    } else {
        for (int e = e0; e < e1; ++e) {
            int c = hst[e];
            hst[e] = run;
            run += c;
        }
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
    int pos = hist[((size_t)which * BH + bh) * tiles * bins +
                   (size_t)key * tiles + tile] +
              rank;
    if (pos < 0 || pos >= N) {
        report(status, kDevSortRange, 0, bh, pos);
        return;
    }
    int32_t *perm = (which ? perm_k : perm_q) + (size_t)bh * N;
    perm[pos] = n;
}

template <typename T, int NS>
cudaError_t launch_hash_t(const Plan &P, const void *q, const void *k,
                          const float *w_sort, uint32_t *keyrank, int *hist,
                          cudaStream_t st) {
    dim3 grid((P.tiles + 1) / 2, P.BH, 2);
    size_t smem = 2 * (size_t)kHashTile * P.d * sizeof(T) +
                  sizeof(float) * (size_t)NS * P.d + sizeof(int) * 8 * P.bins;
    auto kern = k_sort_hash<T, NS>;
    cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize,
                         (int)smem);
    kern<<<grid, kHashTile, smem, st>>>((const T *)q, (const T *)k, w_sort,
                                        P.N, P.d, P.H, P.bins, P.gray,
                                        P.tiles, keyrank, hist);
    return cudaGetLastError();
}

template <int NS>
cudaError_t launch_hash_tma(const Plan &P, const void *q, const void *k,
                            const float *w_sort, uint32_t *keyrank, int *hist,
                            DeviceStatus *status, cudaStream_t st) {
    const uint64_t rows = (uint64_t)P.BH * P.N;
    CUtensorMap tmQ, tmK;
    cudaError_t e =
        make_tma_map_bf16_narrow(&tmQ, q, rows, P.d, kHashCols, kHashBoxRows);
    if (e == cudaSuccess)
        e = make_tma_map_bf16_narrow(&tmK, k, rows, P.d, kHashCols,
                                     kHashBoxRows);
    if (e != cudaSuccess) return e;
    const int quads = (P.tiles + kHashItemTiles - 1) / kHashItemTiles;
    const int items = 2 * P.BH * quads;
    int dev = 0, sms = 148;
    if (cudaGetDevice(&dev) == cudaSuccess)
        cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    const int slots = 2 * sms;  // two CTAs per SM
    const int per = (items + slots - 1) / slots;
    const int grid = (items + per - 1) / per;
    const size_t smem = 512 + (size_t)kHashStages * kHashStageBytes +
                        sizeof(float2) * (size_t)NS * P.d +
                        sizeof(int) * 16 * P.bins;
    auto kern = k_sort_hash_tma<NS>;
    cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize,
                         (int)smem);
    kern<<<grid, kHashThreads, smem, st>>>(tmQ, tmK, w_sort, P.N, P.d, P.H,
                                           P.BH, P.bins, P.gray, P.tiles,
                                           quads, items, per, keyrank, hist,
                                           status);
    return cudaGetLastError();
}

template <typename T>
cudaError_t launch_hash_dtype(const Plan &P, const void *q, const void *k,
                              const float *w_sort, uint32_t *keyrank,
                              int *hist, cudaStream_t st) {
    switch (P.n_s) {
#define ELSAA_NS_CASE(n) \
    case n: return launch_hash_t<T, n>(P, q, k, w_sort, keyrank, hist, st);
        ELSAA_NS_CASE(0) ELSAA_NS_CASE(1) ELSAA_NS_CASE(2) ELSAA_NS_CASE(3)
        ELSAA_NS_CASE(4) ELSAA_NS_CASE(5) ELSAA_NS_CASE(6) ELSAA_NS_CASE(7)
        ELSAA_NS_CASE(8)
#undef ELSAA_NS_CASE
        default: return cudaErrorInvalidValue;
    }
}

}  // namespace

bool hash_tma_supported(const Plan &P) {
    return P.dtype == ELSAA_BF16 && (P.d == 64 || P.d == 128) &&
           P.n_s >= 1 && P.n_s <= 8 && (long)P.BH * P.N >= kHashBoxRows &&
           (long)P.BH * P.N < (1l << 31);
}

cudaError_t launch_sort_hash(const Plan &P, const void *q, const void *k,
                             const float *w_sort, uint32_t *keyrank,
                             int *hist, DeviceStatus *status,
                             cudaStream_t st) {
    if (hash_tma_supported(P)) {
        switch (P.n_s) {
#define ELSAA_NS_CASE(n)                                                   \
    case n:                                                                \
        return launch_hash_tma<n>(P, q, k, w_sort, keyrank, hist, status, st);
            ELSAA_NS_CASE(1) ELSAA_NS_CASE(2) ELSAA_NS_CASE(3)
            ELSAA_NS_CASE(4) ELSAA_NS_CASE(5) ELSAA_NS_CASE(6)
            ELSAA_NS_CASE(7) ELSAA_NS_CASE(8)
#undef ELSAA_NS_CASE
            default: break;
        }
    }
    if (P.dtype == ELSAA_FP32)
        return launch_hash_dtype<float>(P, q, k, w_sort, keyrank, hist, st);
    return launch_hash_dtype<__nv_bfloat16>(P, q, k, w_sort, keyrank, hist,
                                            st);
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
