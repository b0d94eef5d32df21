// Causal ELSAA (Algorithm "Causal ELSAA"): the recursive causal sortLSH
// branch (Algorithm "Causal sortLSH Sparse Exact Attention Branch":
// CausalSparse, SortLSH, MergeLSE) and the chunked causal RACE branch
// (Algorithm "Causal RACE Low-Rank Attention Branch"), bf16 inputs on the
// tensor cores.
//
// The recursion is unrolled. For N = n_leaf 2^Lv (n_leaf <= N0 < 2 n_leaf)
// a row's result is its base segment's exact causal attention, then, from
// the deepest level to the top, MergeLSE with the SortLSH attention of its
// node's future half against the node's past half wherever the row lies in
// a future half. So:
//   k_seg_sort       stable counting sort of each node's future-half query
//                    codes and past-half key codes (codes from the sort hash)
//   k_causal_attn_tc base segments (exact causal attention, 128-row tiles
//                    over 128-key tiles with an online softmax), then one
//                    launch per level, deepest first, for the SortLSH blocks,
//                    merged into the running (O, log d) with MergeLSE
//   race_keys_ws     summaries of segments of G chunks of 128 keys
//   k_seg_offsets    their exclusive prefix over the segments of a head
//   k_causal_scan    per segment, chunk after chunk: the strict prefix
//                    states sA_n, sB_n (offset + the segment's earlier
//                    chunks, accumulated in TMEM; sB_n leaves as bf16)
//   k_causal_race_tc per chunk: inter-chunk readout phi_Q sB_n, intra-chunk
//                    masked products tril(phi_Q phi_K^T) V, then the fusion
//                    of Eq. (5)-(6) with the sparse result.
// The causal RACE result does not depend on the chunk size (exact
// arithmetic); the device uses chunks of 128.
#include "device_common.cuh"
#include "tc_common.cuh"
#include "tc_race.cuh"

namespace elsaa {

namespace {

using namespace tc;

constexpr int kSegThreads = 512;
constexpr int kSegWarps = kSegThreads / 32;
constexpr int kCaThreads = 256;
constexpr float kLog2e = 1.4426950408889634f;
constexpr float kLn2 = 0.6931471805599453f;
constexpr size_t kSmemPerSM = 233472;  // 228 KB of shared memory per SM

// -------------------------------------------------------------- seg sort

// One CTA sorts one segment of m codes stably (equal codes keep increasing
// token order). Segment s of the launch: level l = floor(log2(s + 1)) + 1,
// node j = s + 1 - 2^(l-1); node size n_l = N / 2^(l-1), half m = n_l / 2.
// which 0: the future half's queries (codes of Q), 1: the past half's keys.
// out[l - 1][which][bh][j m + pos] = token index within the head.
__global__ void __launch_bounds__(kSegThreads)
    k_seg_sort(const uint32_t *__restrict__ keyrank, int N, int bins,
               int32_t *__restrict__ perms) {
    __shared__ int cnt[256];
    __shared__ int wc[kSegWarps][256];
    const int s = blockIdx.x, bh = blockIdx.y, which = blockIdx.z;
    const int BH = gridDim.y;
    int l = 1;
    while ((2 << (l - 1)) <= s + 1) ++l;
    const int j = s + 1 - (1 << (l - 1));
    const int n_l = N >> (l - 1), m = n_l >> 1;
    const int base = j * n_l + (which == 0 ? m : 0);
    const uint32_t *codes = keyrank + ((size_t)which * BH + bh) * N + base;
    int32_t *out = perms + (((size_t)(l - 1) * 2 + which) * BH + bh) *
                               (size_t)(N >> 1) +
                   (size_t)j * m;
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    for (int i = tid; i < bins; i += kSegThreads) cnt[i] = 0;
    for (int i = tid; i < kSegWarps * 256; i += kSegThreads)
        (&wc[0][0])[i] = 0;
    __syncthreads();
    for (int i = tid; i < m; i += kSegThreads)
        atomicAdd(&cnt[codes[i] & 0xffffu], 1);
    __syncthreads();
    if (tid == 0) {  // exclusive scan of the histogram
        int run = 0;
        for (int b = 0; b < bins; ++b) {
            const int c = cnt[b];
            cnt[b] = run;
            run += c;
        }
    }
    __syncthreads();
    for (int c0 = 0; c0 < m; c0 += kSegThreads) {
        const int i = c0 + tid;
        const bool in = i < m;
        const int key = in ? (int)(codes[i] & 0xffffu) : -1;
        const unsigned act = __ballot_sync(0xffffffffu, in);
        const unsigned peers = __match_any_sync(0xffffffffu, key) & act;
        const int rank_w = __popc(peers & ((1u << lane) - 1u));
        if (in && rank_w == 0) wc[warp][key] = __popc(peers);
        __syncthreads();
        if (in) {
            int rank = rank_w;
            for (int w = 0; w < warp; ++w) rank += wc[w][key];
            const int pos = cnt[key] + rank;
            if (pos >= 0 && pos < m) out[pos] = base + i;
        }
        __syncthreads();
        for (int b = tid; b < bins; b += kSegThreads) {
            int t = 0;
            for (int w = 0; w < kSegWarps; ++w) {
                t += wc[w][b];
                wc[w][b] = 0;
            }
            cnt[b] += t;
        }
        __syncthreads();
    }
}

// Two fp32 lanes per instruction (fma.rn.f32x2): d = a * b + c lane by lane.
__device__ __forceinline__ unsigned long long ffma2(unsigned long long a,
                                                    unsigned long long b,
                                                    unsigned long long c) {
    unsigned long long d;
    asm("fma.rn.f32x2 %0, %1, %2, %3;" : "=l"(d) : "l"(a), "l"(b), "l"(c));
    return d;
}
__device__ __forceinline__ unsigned long long f2pack(float lo, float hi) {
    unsigned long long d;
    asm("mov.b64 %0, {%1, %2};" : "=l"(d) : "f"(lo), "f"(hi));
    return d;
}
__device__ __forceinline__ void f2unpack(unsigned long long d, float &lo,
                                         float &hi) {
    asm("mov.b64 {%0, %1}, %2;" : "=f"(lo), "=f"(hi) : "l"(d));
}

// ------------------------------------------------------- attention tiles

// One CTA = one tile of 128 query rows and its key tiles, online softmax:
//   mode 0 (base segments): rows leaf n_leaf + 128 qt + [0, 128), key tiles
//          kt = 0..qt of the same segment, the last one masked j <= i;
//          writes (O, log d) of exact causal attention.
//   mode 1 (SortLSH of one level): rows = sorted future-half queries
//          128 qt.. of node j, keys = the node's sorted past-half keys of
//          the same block (b >= 128: b / 128 key tiles; b < 128: one tile,
//          rows and keys paired by block, r / b == c / b); MergeLSE into
//          the running (O, log d).
// Per key tile: MMA S = Q K^T (TMEM [0, 128)); the next K tile's copies
// start at once (K is consumed); CUDA scale, mask, running max and
// P = exp(S - max), packed as bf16 pairs into TMEM over the scores already
// read (keys [64h, 64h + 64) of row half h in columns [64h, 64h + 32));
// MMA P V with P from TMEM (TMEM [128, 128 + D)); the next V tile's copies
// start; CUDA O = O alpha + P V in registers. Two threads per row (TMEM
// lane = row; each takes half of the key columns and half of the output).
// cp.async groups are committed in a fixed order (Q and K0, V0, then per
// tile: next K, next V; empty groups past the last tile), so "all but the
// newest group done" always means the operand about to be used has landed.
template <int D, int MODE>
__global__ void __launch_bounds__(kCaThreads, 2)
    k_causal_attn_tc(const uint16_t *__restrict__ qx,
                     const uint16_t *__restrict__ kx,
                     const uint16_t *__restrict__ vx,
                     const int32_t *__restrict__ permq,
                     const int32_t *__restrict__ permk, int N, int n_leaf,
                     int m, int b, int items, int *__restrict__ next_item,
                     float scale, float eps, float *__restrict__ RO,
                     float *__restrict__ RL, DeviceStatus *status) {
    extern __shared__ unsigned char smem_raw[];
    __shared__ uint64_t mma_bar;
    __shared__ uint32_t tbase;
    __shared__ int abort_flag;
    __shared__ float xm[2][128], xl[2][128];
    __shared__ int qrow_s[128];
    __shared__ int krow_s[2][128];  // MODE 1: key rows of the next tiles
    __shared__ int item_s;
    volatile int *abort = &abort_flag;
    const int tid = threadIdx.x, warp = tid >> 5, lane_id = tid & 31;
    const int half = warp >> 2;
    const int row = (warp & 3) * 32 + lane_id;
    const uint32_t lane = (uint32_t)((warp & 3) * 32) << 16;
    constexpr int DH = D / 2;  // output columns per thread
    constexpr uint32_t kTileB = 128 * D * 2;

    const uint32_t base = align1k(smem_u32(smem_raw));
    const uint32_t sQ = base;
    const uint32_t sK = sQ + kTileB;
    const uint32_t sV = sK + kTileB;

    if (warp == 0) tmem_alloc(&tbase, 256);
    if (tid == 0) {
        mbar_init(&mma_bar, 1);
        abort_flag = 0;
        fence_mbar_init();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tm = tbase;
    uint32_t mph = 0;
    auto mma_done = [&](int site) -> bool {
        if (tid == 0) mma_commit(&mma_bar);
        const bool ok =
            mbar_wait_or_abort(&mma_bar, mph & 1, abort, status, site);
        ++mph;
        tc_fence_after();
        return __syncthreads_and(ok);
    };
    const float sl2 = scale * kLog2e;
    bool ok = true;

    // persistent CTAs take items from a counter (items are numbered longest
    // first, so the take order balances the CTAs)
    while (ok) {
        if (tid == 0) item_s = atomicAdd(next_item, 1);
        __syncthreads();
        const int item = item_s;
        if (item >= items) break;
        // ---- work item
        int bh, qt, nkt, kt0;
        int seg0 = 0;  // MODE 0: first row of the segment (within the head)
        const int32_t *ql = nullptr, *kl = nullptr;
        if (MODE == 0) {
            // item -> (row tile, segment, head), row tiles with the most key
            // tiles first across all segments and heads
            const int nq = n_leaf / 128, nleaves = N / n_leaf;
            const int per = items / nq;  // segments x heads
            qt = nq - 1 - item / per;
            const int rest = item % per;
            const int leaf = rest % nleaves;
            bh = rest / nleaves;
            seg0 = leaf * n_leaf;
            kt0 = 0;
            nkt = qt + 1;
        } else {
            const int tpn = m / 128, nodes = N / (2 * m);
            qt = item % tpn;
            const int rest = item / tpn;
            const int j = rest % nodes;
            bh = rest / nodes;
            ql = permq + (size_t)bh * (N >> 1) + (size_t)j * m;
            kl = permk + (size_t)bh * (N >> 1) + (size_t)j * m;
            if (b >= 128) {
                kt0 = (qt * 128 / b) * (b / 128);
                nkt = b / 128;
            } else {
                kt0 = qt;
                nkt = 1;
            }
        }
        const size_t hN = (size_t)bh * N;
        // key rows of tile kt (tokens within the head); MODE 1 reads them
        // from the level's index list into krow_s[kt & 1] (then a barrier)
        auto stage_rows = [&](int kt) {
            if (MODE == 1 && tid < 128) {
                int t = kl[kt * 128 + tid];
                if (t < 0 || t >= N) {  // read as row 0 (checked: recorded)
#ifdef ELSAA_CHECKED
                    report(status, kDevPermRange, 14, bh, t);
#endif
                    t = 0;
                }
                krow_s[kt & 1][tid] = t;
            }
        };
        auto load_tile = [&](uint32_t dst, const uint16_t *src, int kt) {
            for (int i = tid; i < 128 * (D / 8); i += kCaThreads) {
                const int rr = i / (D / 8), c = i % (D / 8);
                const int t =
                    MODE == 0 ? seg0 + kt * 128 + rr : krow_s[kt & 1][rr];
                cp_async16(dst + panel_offset(rr, c, 128),
                           src + (hN + t) * D + c * 8);
            }
        };
        auto wait_older = [&]() {  // all groups but the newest have landed
            cp_async_wait<1>();
            fence_proxy_async_smem();
            __syncthreads();
        };
        if (tid < 128) {
            int t;
            if (MODE == 0) {
                t = seg0 + qt * 128 + tid;
            } else {
                t = ql[qt * 128 + tid];
                if (t < 0 || t >= N) {  // read as row 0 (checked: recorded)
#ifdef ELSAA_CHECKED
                    report(status, kDevPermRange, 15, bh, t);
#endif
                    t = 0;
                }
            }
            qrow_s[tid] = t;
        }
        stage_rows(kt0);
        __syncthreads();
        for (int i = tid; i < 128 * (D / 8); i += kCaThreads) {
            const int rr = i / (D / 8), c = i % (D / 8);
            cp_async16(sQ + panel_offset(rr, c, 128),
                       qx + (hN + qrow_s[rr]) * D + c * 8);
        }
        load_tile(sK, kx, kt0);
        cp_async_commit();
        load_tile(sV, vx, kt0);
        cp_async_commit();

        unsigned long long o_acc[DH / 2];  // output pairs (f32x2)
#pragma unroll
        for (int j = 0; j < DH / 2; ++j) o_acc[j] = 0ull;
        float mrun = -INFINITY, lrun = 0.0f;  // log2 domain max, sum
        for (int it = 0; it < nkt && ok; ++it) {
            const int kt = kt0 + it;
            wait_older();  // K of this tile
            if (tid == 0) {
                tc_fence_after();
                const uint32_t id = idesc_bf16(128, 128, false, false);
#pragma unroll
                for (int k = 0; k < D / 16; ++k)
                    mma_ss(tm,
                           smem_desc(sQ + (k >> 2) * 16384 + (k & 3) * 32, 16,
                                     1024),
                           smem_desc(sK + (k >> 2) * 16384 + (k & 3) * 32, 16,
                                     1024),
                           id, k > 0);
            }
            if (!(ok = mma_done(120))) break;
            if (it + 1 < nkt) {
                if (MODE == 1) {
                    stage_rows(kt + 1);
                    __syncthreads();
                }
                load_tile(sK, kx, kt + 1);
            }
            cp_async_commit();

            // ---- running max (two 32-column passes over the raw scores;
            // the scale is positive), then P = 2^(scale log2e S - max)
            // packed over the scores already read. Masks only on the
            // diagonal tile (MODE 0) or with several blocks per tile
            // (MODE 1, b < 128).
            const bool any_mask = MODE == 0 ? kt == qt : b < 128;
            // kept key columns [klo, khi) of this row: the causal prefix of
            // the diagonal tile, or the row's own block
            const int klo = MODE == 0 ? 0 : (row / b) * b;
            const int khi = MODE == 0 ? row + 1 : klo + b;
            auto keep = [&](int c) -> bool { return c >= klo && c < khi; };
            float mx = -INFINITY;
#pragma unroll
            for (int j0 = 0; j0 < 64; j0 += 32) {
                uint32_t v[32];
                tmem_ld32(tm + lane + 64 * half + j0, v);
                tmem_wait_ld();
                if (any_mask) {
#pragma unroll
                    for (int j = 0; j < 32; ++j)
                        if (keep(64 * half + j0 + j))
                            mx = fmaxf(mx, __uint_as_float(v[j]));
                } else {
#pragma unroll
                    for (int j = 0; j < 32; ++j)
                        mx = fmaxf(mx, __uint_as_float(v[j]));
                }
            }
            xm[half][row] = mx * sl2;  // -inf stays -inf
            __syncthreads();
            const float mnew = fmaxf(mrun, fmaxf(xm[0][row], xm[1][row]));
            const float alpha = ex2_approx(mrun - mnew);  // 0 on tile 0
            const unsigned long long sl2x2 = f2pack(sl2, sl2);
            const unsigned long long nm2 = f2pack(-mnew, -mnew);
            const unsigned long long one2 = f2pack(1.0f, 1.0f);
            unsigned long long ls2 = 0ull;
#pragma unroll
            for (int j0 = 0; j0 < 64; j0 += 32) {
                uint32_t v[32];
                tmem_ld32(tm + lane + 64 * half + j0, v);
                tmem_wait_ld();
                uint32_t pk[16];
#pragma unroll
                for (int j = 0; j < 32; j += 2) {
                    float x0, x1;
                    f2unpack(ffma2(f2pack(__uint_as_float(v[j]),
                                          __uint_as_float(v[j + 1])),
                                   sl2x2, nm2),
                             x0, x1);
                    float a0 = ex2_approx(x0);
                    float a1 = ex2_approx(x1);
                    if (any_mask) {
                        a0 = keep(64 * half + j0 + j) ? a0 : 0.0f;
                        a1 = keep(64 * half + j0 + j + 1) ? a1 : 0.0f;
                    }
                    ls2 = ffma2(f2pack(a0, a1), one2, ls2);
                    pk[j >> 1] = pack_bf16x2(a0, a1);
                }
                // over scores of this thread's half already read
                tmem_st16(tm + lane + 64 * half + j0 / 2, pk);
            }
            tmem_wait_st();
            float lsa, lsb;
            f2unpack(ls2, lsa, lsb);
            xl[half][row] = lsa + lsb;
            tc_fence_before();
            __syncthreads();
            lrun = lrun * alpha + xl[0][row] + xl[1][row];
            mrun = mnew;

            // ---- P V (P from TMEM: keys 16 k.. of half k / 4 sit at
            // columns 64 (k / 4) + 8 (k % 4))
            wait_older();  // V of this tile
            if (tid == 0) {
                tc_fence_after();
                const uint32_t id = idesc_bf16(128, D, false, true);
#pragma unroll
                for (int k = 0; k < 8; ++k)
                    mma_ts(tm + 128,
                           tm + (uint32_t)(64 * (k >> 2) + 8 * (k & 3)),
                           smem_desc(sV + k * 2048, 16384, 1024), id, k > 0);
            }
            if (!(ok = mma_done(121))) break;
            if (it + 1 < nkt) load_tile(sV, vx, kt + 1);
            cp_async_commit();
            const unsigned long long al2 = f2pack(alpha, alpha);
#pragma unroll
            for (int c = 0; c < DH; c += 32) {
                uint32_t v[32];
                tmem_ld32(tm + lane + 128 + half * DH + c, v);
                tmem_wait_ld();
#pragma unroll
                for (int j = 0; j < 32; j += 2)
                    o_acc[(c + j) / 2] =
                        ffma2(o_acc[(c + j) / 2], al2,
                              f2pack(__uint_as_float(v[j]),
                                     __uint_as_float(v[j + 1])));
            }
            tc_fence_before();
        }
        cp_async_wait<0>();
        __syncthreads();  // the next item's copies reuse every buffer
        if (!ok) break;

        // ---- O = sum e^z V / (sum e^z + eps), log d (natural log)
        const float logd = (mrun + log2f(lrun)) * kLn2;
        const float inv = 1.0f / (lrun + eps * ex2_approx(-mrun));
        const size_t tok = hN + qrow_s[row];
        float *o = RO + tok * D + half * DH;
        float ld_new = logd;
        float of[DH];
#pragma unroll
        for (int j = 0; j < DH / 2; ++j) f2unpack(o_acc[j], of[2 * j], of[2 * j + 1]);
        if (MODE == 0) {
#pragma unroll
            for (int j = 0; j < DH; j += 4)
                *reinterpret_cast<float4 *>(o + j) =
                    make_float4(of[j] * inv, of[j + 1] * inv,
                                of[j + 2] * inv, of[j + 3] * inv);
            if (half == 0) RL[tok] = logd;
        } else {
            // MergeLSE(running = diag, this = off)
            const float ld1 = RL[tok];
            const float mu = fmaxf(ld1, logd);
            const float w1 = __expf(ld1 - mu), w2 = __expf(logd - mu);
            const float ssum = w1 + w2;
            const float r = 1.0f / (ssum + eps);
            const float c1 = w1 * r, c2 = w2 * inv * r;
#pragma unroll
            for (int j = 0; j < DH; j += 4) {
                float4 a = *reinterpret_cast<float4 *>(o + j);
                a.x = c1 * a.x + c2 * of[j];
                a.y = c1 * a.y + c2 * of[j + 1];
                a.z = c1 * a.z + c2 * of[j + 2];
                a.w = c1 * a.w + c2 * of[j + 3];
                *reinterpret_cast<float4 *>(o + j) = a;
            }
            ld_new = mu + __logf(ssum + eps);
        }
        __syncthreads();  // qrow_s is rewritten by the next item; both
                          // halves read RL before it changes
        if (MODE == 1 && half == 0) RL[tok] = ld_new;
    }
    cp_async_wait<0>();
    tc_fence_before();
    __syncthreads();
    if (warp == 0) tmem_dealloc(tm, 256);
}

// ---------------------------------------------------- RACE prefix states

// Segment offsets in place: part[bh][s] (segment totals B, A) becomes the
// sum over the segments before s (fp32).
__global__ void k_seg_offsets(float *__restrict__ part, int nseg, int r,
                              int d) {
    const int bh = blockIdx.y;
    const size_t per = (size_t)r * d + r;
    const size_t i = (size_t)blockIdx.x * blockDim.x + threadIdx.x;
    if (i >= per) return;
    float *p = part + (size_t)bh * nseg * per + i;
    float run = 0.0f;
    for (int s0 = 0; s0 < nseg; s0 += 8) {  // eight loads in flight
        float v[8];
#pragma unroll
        for (int j = 0; j < 8; ++j)
            v[j] = s0 + j < nseg ? p[(size_t)(s0 + j) * per] : 0.0f;
#pragma unroll
        for (int j = 0; j < 8; ++j)
            if (s0 + j < nseg) {
                p[(size_t)(s0 + j) * per] = run;
                run += v[j];
            }
    }
}

// Prefix states of one segment of G chunks (128 keys each), in order: the
// state starts at the segment's offset (the sum over earlier segments) and
// grows by each chunk's [B_n | A_n] = phi(K_n)^T [V_n | 1]; before chunk n
// is added, sB_n (bf16) and sA_n (fp32) are written. One CTA per (head,
// segment), 256 threads, TMEM: accumulator M-tile m at m (D + 16) (B in the
// first D columns, A repeated in the next 16), projections after them.
template <int D, int L>
__global__ void __launch_bounds__(kCaThreads, 1)
    k_causal_scan(const uint16_t *__restrict__ kx,
                  const uint16_t *__restrict__ vx,
                  const uint16_t *__restrict__ w_bf16,
                  const float *__restrict__ offs, int N, int H, int nseg,
                  int G, float beta, uint16_t *__restrict__ sBh,
                  float *__restrict__ sA, DeviceStatus *status) {
    constexpr int R = 16, Gb = 4;
    constexpr int r = L * R, Lg = L * Gb;
    constexpr int Lg_pad = (Lg + 15) / 16 * 16;
    constexpr int r_pad = r < 128 ? 128 : r;
    constexpr int nM = r_pad / 128;
    constexpr int TPT = L / 2;  // tables per thread (two threads per key)
    constexpr uint32_t kAccN = D + 16;
    constexpr uint32_t kColP = nM * kAccN;  // projections
    constexpr uint32_t kTileB = 128 * D * 2;
    extern __shared__ unsigned char smem_raw[];
    __shared__ uint64_t mma_bar;
    __shared__ uint32_t tbase;
    __shared__ int abort_flag;
    volatile int *abort = &abort_flag;
    const int tid = threadIdx.x, warp = tid >> 5, lane_id = tid & 31;
    const int half = warp >> 2;
    const int row = (warp & 3) * 32 + lane_id;
    const uint32_t lane = (uint32_t)((warp & 3) * 32) << 16;

    const uint32_t base = align1k(smem_u32(smem_raw));
    const uint32_t sK = base;                    // [128 x D]
    const uint32_t sV = sK + kTileB;             // [128 x D], then ones
    const uint32_t sW = sV + kTileB + 16384;     // [Lg_pad x D]
    const uint32_t sPhi = sW + align1k((uint32_t)Lg_pad * D * 2);  // [128 x r_pad]

    const int seg = blockIdx.x % nseg, bh = blockIdx.x / nseg;
    const int h = bh % H;
    const int nc = N / 128;
    const size_t per = (size_t)r * D + r;
    const float *off = offs + ((size_t)bh * nseg + seg) * per;

    if (warp == 0) tmem_alloc(&tbase, 512);
    if (tid == 0) {
        mbar_init(&mma_bar, 1);
        abort_flag = 0;
        fence_mbar_init();
    }
    for (int i = tid; i < 16384 / 16; i += kCaThreads)  // bf16 ones
        asm volatile("st.shared.v4.b32 [%0], {%1, %1, %1, %1};" ::"r"(
                         sV + kTileB + i * 16),
                     "r"(0x3F803F80u)
                     : "memory");
    if (r < r_pad)  // buckets past r stay zero
        for (int i = tid; i < 128 * (r_pad - r) / 8; i += kCaThreads) {
            const int rr = i / ((r_pad - r) / 8), c = i % ((r_pad - r) / 8);
            st_shared_zero16(sPhi + panel_offset(rr, r / 8 + c, 128));
        }
    for (int i = tid; i < Lg_pad * (D / 8); i += kCaThreads) {
        const int rr = i / (D / 8), c = i % (D / 8);
        cp_async16(sW + panel_offset(rr, c, Lg_pad),
                   w_bf16 + ((size_t)h * Lg_pad + rr) * D + c * 8);
    }
    auto load_k = [&](int n) {
        const size_t r0 = (size_t)bh * N + (size_t)n * 128;
        for (int i = tid; i < 128 * (D / 8); i += kCaThreads) {
            const int rr = i / (D / 8), c = i % (D / 8);
            cp_async16(sK + panel_offset(rr, c, 128), kx + (r0 + rr) * D + c * 8);
        }
    };
    auto load_v = [&](int n) {
        const size_t r0 = (size_t)bh * N + (size_t)n * 128;
        for (int i = tid; i < 128 * (D / 8); i += kCaThreads) {
            const int rr = i / (D / 8), c = i % (D / 8);
            cp_async16(sV + panel_offset(rr, c, 128), vx + (r0 + rr) * D + c * 8);
        }
    };
    const int n0 = seg * G;
    load_k(n0);
    load_v(n0);
    cp_async_commit();
    fence_proxy_async_smem();
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tm = tbase;
    uint32_t mph = 0;
    auto mma_done = [&](int site) -> bool {
        if (tid == 0) mma_commit(&mma_bar);
        const bool ok =
            mbar_wait_or_abort(&mma_bar, mph & 1, abort, status, site);
        ++mph;
        tc_fence_after();
        return __syncthreads_and(ok);
    };
    // The accumulator starts at the segment's offset (written into TMEM by
    // the lanes that own the buckets), so every state is read from TMEM:
    // thread (lane, half) owns buckets m 128 + lane of M-tiles m = half,
    // half + 2, ...
    for (int m = half; m < nM; m += 2) {
        const int bk = m * 128 + row;
        const float *ob = off + (size_t)(bk < r ? bk : 0) * D;
#pragma unroll
        for (int c = 0; c < D; c += 32) {
            uint32_t v[32];
#pragma unroll
            for (int j = 0; j < 32; j += 4) {
                const float4 a = *reinterpret_cast<const float4 *>(ob + c + j);
                v[j] = __float_as_uint(bk < r ? a.x : 0.0f);
                v[j + 1] = __float_as_uint(bk < r ? a.y : 0.0f);
                v[j + 2] = __float_as_uint(bk < r ? a.z : 0.0f);
                v[j + 3] = __float_as_uint(bk < r ? a.w : 0.0f);
            }
            tmem_st32(tm + lane + m * kAccN + c, v);
        }
        uint32_t a16[16];
        const float av = bk < r ? off[(size_t)r * D + bk] : 0.0f;
#pragma unroll
        for (int j = 0; j < 16; ++j) a16[j] = __float_as_uint(av);
        tmem_st16(tm + lane + m * kAccN + D, a16);
    }
    tmem_wait_st();
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    // sB_n (bf16), sA_n = the accumulated state
    auto write_state = [&](int n) {
        const size_t cidx = (size_t)bh * nc + n;
        for (int m = half; m < nM; m += 2) {
            const int bk = m * 128 + row;
            uint16_t *out = sBh + (cidx * r + (bk < r ? bk : 0)) * D;
#pragma unroll
            for (int c = 0; c < D; c += 32) {
                uint32_t v[32];
                tmem_ld32(tm + lane + m * kAccN + c, v);
                tmem_wait_ld();
                if (bk < r) {
#pragma unroll
                    for (int j = 0; j < 32; j += 8) {
                        uint4 pk;
                        pk.x = pack_bf16x2(__uint_as_float(v[j]),
                                           __uint_as_float(v[j + 1]));
                        pk.y = pack_bf16x2(__uint_as_float(v[j + 2]),
                                           __uint_as_float(v[j + 3]));
                        pk.z = pack_bf16x2(__uint_as_float(v[j + 4]),
                                           __uint_as_float(v[j + 5]));
                        pk.w = pack_bf16x2(__uint_as_float(v[j + 6]),
                                           __uint_as_float(v[j + 7]));
                        *reinterpret_cast<uint4 *>(out + c + j) = pk;
                    }
                }
            }
            uint32_t v16[16];
            tmem_ld16(tm + lane + m * kAccN + D, v16);
            tmem_wait_ld();
            if (bk < r) sA[cidx * r + bk] = __uint_as_float(v16[0]);
        }
    };
    write_state(n0);

    bool ok = true;
    for (int c = 0; c < G && ok; ++c) {
        const int n = n0 + c;
        cp_async_wait<0>();
        fence_proxy_async_smem();
        __syncthreads();
        if (tid == 0) {  // projections U = K W^T
            tc_fence_after();
            const uint32_t id = idesc_bf16(128, Lg_pad, false, false);
#pragma unroll
            for (int k = 0; k < D / 16; ++k)
                mma_ss(tm + kColP,
                       smem_desc(sK + (k >> 2) * 16384 + (k & 3) * 32, 16, 1024),
                       smem_desc(sW + (k >> 2) * Lg_pad * 128 + (k & 3) * 32,
                                 16, 1024),
                       id, k > 0);
        }
        if (!(ok = mma_done(140))) break;
        if (c + 1 < G) load_k(n + 1);  // this chunk's K is consumed
        // features of this thread's tables
#pragma unroll
        for (int t = 0; t < TPT; ++t) {
            const int tbl = half * TPT + t;
            uint32_t u4[16];
            tmem_ld16(tm + lane + kColP + (tbl * Gb) / 16 * 16, u4);
            tmem_wait_ld();
            float sp[Gb];
#pragma unroll
            for (int bb = 0; bb < Gb; ++bb) {
                // column of bit bb of table tbl within the 16 loaded; the
                // half-dependent part is 0 or 8 (no dynamic indexing)
                const int i0 = (t * Gb) % 16 + bb;
                const uint32_t u =
                    (TPT * Gb) % 16 == 0 ? u4[i0]
                                         : (half ? u4[(i0 + 8) & 15] : u4[i0]);
                sp[bb] = fmaf(0.5f,
                              tanh_approx(beta * tanh_approx(__uint_as_float(u))),
                              0.5f);
            }
            float phi[R];
            table_phi<Gb>(sp, phi);
            st_shared_bf16x8(sPhi + panel_offset(row, tbl * 2, 128), phi);
            st_shared_bf16x8(sPhi + panel_offset(row, tbl * 2 + 1, 128), phi + 8);
        }
        fence_proxy_async_smem();
        tc_fence_before();
        __syncthreads();
        if (tid == 0) {  // state += phi^T [V | 1]
            tc_fence_after();
            const uint32_t id = idesc_bf16(128, D + 16, true, true);
            for (int m = 0; m < nM; ++m)
#pragma unroll
                for (int k = 0; k < 8; ++k)
                    mma_ss(tm + m * kAccN,
                           smem_desc(sPhi + 2 * m * 16384 + k * 2048, 16384, 1024),
                           smem_desc(sV + k * 2048, 16384, 1024), id, 1u);
        }
        if (!(ok = mma_done(141))) break;
        if (c + 1 < G) {
            load_v(n + 1);  // this chunk's V is consumed
            cp_async_commit();
            write_state(n + 1);
        }
        tc_fence_before();
        __syncthreads();
    }
    cp_async_wait<0>();
    tc_fence_before();
    __syncthreads();
    if (warp == 0) tmem_dealloc(tm, 512);
}

// ----------------------------------------------- causal RACE + fusion

// One CTA = one chunk of 128 tokens of one head (original order):
//   MMA  U_Q = Q W^T, U_K = K W^T
//   per 128-bucket group h: CUDA phi_Q, phi_K of the group's tables and
//        phi_Q . sA_n; MMA S += phi_Q phi_K^T, Num += phi_Q sB_n
//   CUDA P = tril(S) (bf16), row sums
//   MMA  Num += P V
//   CUDA O_lr = Num / L / (Den / L + eps), then Eq. (5)-(6) with the
//        sparse branch's (O_s, log d_s).
// TMEM: U_Q [0, 64), U_K [64, 128), S [128, 256), Num [256, 256 + D).
template <int D, int L>
__global__ void __launch_bounds__(kCaThreads, 1)
    k_causal_race_tc(const uint16_t *__restrict__ qx,
                     const uint16_t *__restrict__ kx,
                     const uint16_t *__restrict__ vx,
                     const uint16_t *__restrict__ w_bf16,
                     const uint16_t *__restrict__ sBh,
                     const float *__restrict__ sAg, const float *__restrict__ RO,
                     const float *__restrict__ RL,
                     const float *__restrict__ lambda_tok,
                     const float *__restrict__ gates, int N, int H, float beta,
                     float eps, float lambda, int mode,
                     uint16_t *__restrict__ ox, float *__restrict__ o32,
                     float *__restrict__ log_ds_out,
                     float *__restrict__ dlr_out, float *__restrict__ m_out,
                     DeviceStatus *status) {
    constexpr int R = 16, G = 4;
    constexpr int r = L * R, Lg = L * G;
    constexpr int Lg_pad = (Lg + 15) / 16 * 16;
    constexpr int RB = r < 128 ? r : 128;  // buckets per group
    constexpr int NG = r / RB;             // groups
    constexpr int TPT = RB / R / 2;        // tables per thread and group
    constexpr int DH = D / 2;
    constexpr uint32_t kTileB = 128 * D * 2;
    extern __shared__ unsigned char smem_raw[];
    __shared__ uint64_t mma_bar;
    __shared__ uint32_t tbase;
    __shared__ int abort_flag;
    __shared__ float xd[2][128];
    volatile int *abort = &abort_flag;
    const int tid = threadIdx.x, warp = tid >> 5, lane_id = tid & 31;
    const int half = warp >> 2;
    const int row = (warp & 3) * 32 + lane_id;
    const uint32_t lane = (uint32_t)((warp & 3) * 32) << 16;

    const uint32_t base = align1k(smem_u32(smem_raw));
    const uint32_t sQ = base;            // Q, then phi_Q of a group, then P
    const uint32_t sK = sQ + 32768;      // K, then phi_K of a group
    const uint32_t sB = sK + 32768;      // sB_n [r x D]
    const uint32_t sV = sB + (uint32_t)r * D * 2;
    const uint32_t sW = sV + kTileB;     // [Lg_pad x D]
    const uint32_t sAo = sW + (uint32_t)Lg_pad * D * 2;  // fp32 sA_n [r]
    const float *sAf =
        reinterpret_cast<const float *>(smem_raw + (sAo - smem_u32(smem_raw)));

    const int nc = N / 128;
    const int bh = blockIdx.x / nc, n = blockIdx.x % nc;
    const int h = bh % H;
    const size_t row0 = (size_t)bh * N + (size_t)n * 128;

    if (warp == 0) tmem_alloc(&tbase, 512);
    if (tid == 0) {
        mbar_init(&mma_bar, 1);
        abort_flag = 0;
        fence_mbar_init();
    }
    // two copy groups: what the projections and features need (Q, K,
    // planes, sA_n), then what the products after them need (V, sB_n)
    for (int i = tid; i < 128 * (D / 8); i += kCaThreads) {
        const int rr = i / (D / 8), c = i % (D / 8);
        const size_t o = (row0 + rr) * D + c * 8;
        cp_async16(sQ + panel_offset(rr, c, 128), qx + o);
        cp_async16(sK + panel_offset(rr, c, 128), kx + o);
    }
    for (int i = tid; i < Lg_pad * (D / 8); i += kCaThreads) {
        const int rr = i / (D / 8), c = i % (D / 8);
        cp_async16(sW + panel_offset(rr, c, Lg_pad),
                   w_bf16 + ((size_t)h * Lg_pad + rr) * D + c * 8);
    }
    const size_t cidx = (size_t)bh * nc + n;
    for (int i = tid; i < r / 4; i += kCaThreads)
        cp_async16(sAo + 16 * i, sAg + cidx * r + 4 * i);
    cp_async_commit();
    for (int i = tid; i < 128 * (D / 8); i += kCaThreads) {
        const int rr = i / (D / 8), c = i % (D / 8);
        cp_async16(sV + panel_offset(rr, c, 128), vx + (row0 + rr) * D + c * 8);
    }
    for (int i = tid; i < r * (D / 8); i += kCaThreads) {
        const int rr = i / (D / 8), c = i % (D / 8);
        cp_async16(sB + panel_offset(rr, c, r),
                   sBh + (cidx * r + rr) * D + c * 8);
    }
    cp_async_commit();
    cp_async_wait<1>();
    fence_proxy_async_smem();
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tm = tbase;
    uint32_t mph = 0;
    auto mma_done = [&](int site) -> bool {
        if (tid == 0) mma_commit(&mma_bar);
        const bool ok =
            mbar_wait_or_abort(&mma_bar, mph & 1, abort, status, site);
        ++mph;
        tc_fence_after();
        return __syncthreads_and(ok);
    };

    bool ok = true;
    // ---- projections
    if (tid == 0) {
        const uint32_t id = idesc_bf16(128, Lg_pad, false, false);
#pragma unroll
        for (int k = 0; k < D / 16; ++k) {
            const uint32_t oa = (k >> 2) * 16384 + (k & 3) * 32;
            const uint64_t bw =
                smem_desc(sW + (k >> 2) * Lg_pad * 128 + (k & 3) * 32, 16,
                          1024);
            mma_ss(tm, smem_desc(sQ + oa, 16, 1024), bw, id, k > 0);
            mma_ss(tm + 64, smem_desc(sK + oa, 16, 1024), bw, id, k > 0);
        }
    }
    ok = mma_done(130);

    float den_inter = 0.0f;
    for (int g = 0; g < NG && ok; ++g) {
        // features of this thread's tables in group g (the group's
        // projections are TMEM columns [32 g, 32 g + RB / 4); with 128
        // buckets per group each half's 16 columns load alone, with 64 the
        // two halves share one 16-column load)
        uint32_t uq[16], uk[16];
        const uint32_t c0 = 32 * g + (RB == 128 ? 16 * half : 0);
        tmem_ld16(tm + lane + c0, uq);
        tmem_ld16(tm + lane + 64 + c0, uk);
        tmem_wait_ld();
        auto pick = [&](const uint32_t(&u)[16], int i) -> float {
            if (RB == 128) return __uint_as_float(u[i]);
            return __uint_as_float(half ? u[(8 + i) & 15] : u[i]);
        };
#pragma unroll
        for (int t = 0; t < TPT; ++t) {
            const int tl = half * TPT + t;       // table within the group
            const int tbl = g * (RB / R) + tl;  // table
            // per-bit factors sigma(2 beta tanh u) = 1/2 + tanh(beta tanh u)/2
            float spq[G], spk[G];
#pragma unroll
            for (int bb = 0; bb < G; ++bb) {
                spq[bb] = fmaf(0.5f,
                               tanh_approx(beta * tanh_approx(
                                                      pick(uq, t * G + bb))),
                               0.5f);
                spk[bb] = fmaf(0.5f,
                               tanh_approx(beta * tanh_approx(
                                                      pick(uk, t * G + bb))),
                               0.5f);
            }
            float pq[R], pk[R];
            table_phi<G>(spq, pq);
            table_phi<G>(spk, pk);
#pragma unroll
            for (int rr = 0; rr < R; ++rr)
                den_inter = fmaf(pq[rr], sAf[tbl * R + rr], den_inter);
            const int col = tl * R;  // bucket within the group
            st_shared_bf16x8(sQ + panel_offset(row, col / 8, 128), pq);
            st_shared_bf16x8(sQ + panel_offset(row, col / 8 + 1, 128), pq + 8);
            st_shared_bf16x8(sK + panel_offset(row, col / 8, 128), pk);
            st_shared_bf16x8(sK + panel_offset(row, col / 8 + 1, 128), pk + 8);
        }
        if (g == 0) cp_async_wait<0>();  // V and sB_n
        fence_proxy_async_smem();
        tc_fence_before();
        __syncthreads();
        if (tid == 0) {
            tc_fence_after();
            const uint32_t id_s = idesc_bf16(128, 128, false, false);
            const uint32_t id_n = idesc_bf16(128, D, false, true);
#pragma unroll
            for (int k = 0; k < RB / 16; ++k) {
                const uint32_t oa = (k >> 2) * 16384 + (k & 3) * 32;
                mma_ss(tm + 128, smem_desc(sQ + oa, 16, 1024),
                       smem_desc(sK + oa, 16, 1024), id_s, (g > 0 || k > 0));
                mma_ss(tm + 256, smem_desc(sQ + oa, 16, 1024),
                       smem_desc(sB + (uint32_t)(g * RB + 16 * k) * 128,
                                 (uint32_t)r * 128, 1024),
                       id_n, (g > 0 || k > 0));
            }
        }
        ok = mma_done(131);
    }

    // the sparse result of the chunk's rows into the consumed sB_n space
    // (fp32 rows, 16-byte chunk c of row i at c ^ (i & 7)), read back by
    // the epilogue; with r < 256 the epilogue reads it from global memory
    constexpr bool kStageRO = r >= 256;
    if (kStageRO && ok) {
        for (int i = tid; i < 128 * (D / 4); i += kCaThreads) {
            const int rr = i / (D / 4), c = i % (D / 4);
            cp_async16(sB + rr * (D * 4) + ((c ^ (rr & 7)) << 4),
                       RO + (row0 + rr) * D + c * 4);
        }
        cp_async_commit();
    }

    // ---- P = tril(S): row i keeps keys j <= i of the chunk
    float dintra = 0.0f;
    if (ok) {
        float s[64];
        uint32_t v[32];
        tmem_ld32(tm + lane + 128 + 64 * half, v);
        tmem_wait_ld();
#pragma unroll
        for (int j = 0; j < 32; ++j) s[j] = __uint_as_float(v[j]);
        tmem_ld32(tm + lane + 128 + 64 * half + 32, v);
        tmem_wait_ld();
#pragma unroll
        for (int j = 0; j < 32; ++j) s[32 + j] = __uint_as_float(v[j]);
#pragma unroll
        for (int j = 0; j < 64; ++j) {
            s[j] = (64 * half + j <= row) ? s[j] : 0.0f;
            dintra += s[j];
        }
#pragma unroll
        for (int q = 0; q < 8; ++q)
            st_shared_bf16x8(sQ + panel_offset(row, 8 * half + q, 128),
                             s + 8 * q);
        fence_proxy_async_smem();
        tc_fence_before();
    }
    xd[half][row] = den_inter + dintra;
    __syncthreads();
    if (ok && tid == 0) {
        tc_fence_after();
        const uint32_t id = idesc_bf16(128, D, false, true);
#pragma unroll
        for (int k = 0; k < 8; ++k)
            mma_ss(tm + 256,
                   smem_desc(sQ + (k >> 2) * 16384 + (k & 3) * 32, 16, 1024),
                   smem_desc(sV + k * 2048, 16384, 1024), id, 1u);
    }
    if (ok) ok = mma_done(132);
    if (kStageRO) {
        cp_async_wait<0>();
        __syncthreads();
    }

    if (ok) {
        const float invL = 1.0f / (float)L;
        const float den = (xd[0][row] + xd[1][row]) * invL;
        const float rl = 1.0f / (den + eps);
        const size_t tok = row0 + row;
        const float log_ds = RL[tok];
        const float lam = lambda_tok ? lambda_tok[tok] : lambda;
        const float gs = gates ? gates[2 * tok] : 1.0f;
        const float gl = gates ? gates[2 * tok + 1] : 1.0f;
        const float mm = fusion_multiplier(log_ds, lam, den, eps, mode);
        const float cs = gs * mm, cl = gl * invL * rl;
        const float4 *os =
            reinterpret_cast<const float4 *>(RO + tok * D + half * DH);
        uint16_t *o = ox + tok * D + half * DH;
#pragma unroll
        for (int c = 0; c < DH; c += 32) {
            uint32_t v[32];
            tmem_ld32(tm + lane + 256 + half * DH + c, v);
            tmem_wait_ld();
#pragma unroll
            for (int j = 0; j < 32; j += 8) {
                float4 s0, s1;
                if (kStageRO) {
                    const int c0 = (half * DH + c + j) / 4;  // 16-byte chunk
                    const unsigned char *rb =
                        smem_raw + (sB - smem_u32(smem_raw)) + row * (D * 4);
                    s0 = *reinterpret_cast<const float4 *>(
                        rb + ((c0 ^ (row & 7)) << 4));
                    s1 = *reinterpret_cast<const float4 *>(
                        rb + (((c0 + 1) ^ (row & 7)) << 4));
                } else {
                    s0 = os[(c + j) / 4];
                    s1 = os[(c + j) / 4 + 1];
                }
                const float sv[8] = {s0.x, s0.y, s0.z, s0.w,
                                     s1.x, s1.y, s1.z, s1.w};
                float y[8];
#pragma unroll
                for (int e = 0; e < 8; ++e)
                    y[e] = cs * sv[e] + cl * __uint_as_float(v[j + e]);
                if (o32) {  // fp32 output: two 16-byte stores
                    float4 *dst = reinterpret_cast<float4 *>(
                        o32 + tok * D + half * DH + c + j);
                    dst[0] = make_float4(y[0], y[1], y[2], y[3]);
                    dst[1] = make_float4(y[4], y[5], y[6], y[7]);
                    continue;
                }
                uint4 pk;
                pk.x = pack_bf16x2(y[0], y[1]);
                pk.y = pack_bf16x2(y[2], y[3]);
                pk.z = pack_bf16x2(y[4], y[5]);
                pk.w = pack_bf16x2(y[6], y[7]);
                *reinterpret_cast<uint4 *>(o + c + j) = pk;
            }
        }
        if (half == 0) {
            if (log_ds_out) log_ds_out[tok] = log_ds;
            if (dlr_out) dlr_out[tok] = den;
            if (m_out) m_out[tok] = mm;
        }
    }
    tc_fence_before();
    __syncthreads();
    if (warp == 0) tmem_dealloc(tm, 512);
}

}  // namespace

// ------------------------------------------------------------------ host

bool causal_tc_supported(const Plan &P, int n_leaf) {
    if (P.dtype != ELSAA_BF16 || P.impl != 2) return false;
    if (P.d != 64 && P.d != 128) return false;
    if (P.gamma != 4 || !(P.L == 4 || P.L == 8 || P.L == 16)) return false;
    if (n_leaf % 128 != 0 || P.N % 128 != 0) return false;
    if (!(P.b == 32 || P.b == 64 || P.b == 128 || P.b == 256)) return false;
    if (n_leaf != P.N && n_leaf % P.b != 0) return false;
    return true;
}

size_t causal_attn_smem(int d) { return 1024 + (size_t)3 * 128 * d * 2; }

size_t causal_race_smem(const Plan &P) {
    const size_t lg_pad = ((size_t)P.L * 4 + 15) / 16 * 16;
    return 1024 + 65536 + (size_t)P.r * P.d * 2 + (size_t)128 * P.d * 2 +
           lg_pad * P.d * 2 + (size_t)P.r * 4;
}

cudaError_t launch_seg_sort(const Plan &P, int Lv, const uint32_t *keyrank,
                            int32_t *perms, cudaStream_t st) {
    if (Lv == 0) return cudaSuccess;
    dim3 grid((1u << Lv) - 1, P.BH, 2);
    k_seg_sort<<<grid, kSegThreads, 0, st>>>(keyrank, P.N, P.bins, perms);
    return cudaGetLastError();
}

// mode 0: base segments of n_leaf rows; mode 1: SortLSH blocks of level
// `level` (1 = top) whose halves hold m = N / 2^level rows.
cudaError_t launch_causal_attn(const Plan &P, int mode, int n_leaf, int level,
                               const void *q, const void *k, const void *v,
                               const int32_t *perms, int *next_item, float *RO,
                               float *RL, DeviceStatus *status,
                               cudaStream_t st) {
    int items, m = 0;
    const int32_t *pq = nullptr, *pk = nullptr;
    if (mode == 0) {
        items = P.BH * (P.N / n_leaf) * (n_leaf / 128);
    } else {
        m = P.N >> level;
        items = P.BH * (P.N / (2 * m)) * (m / 128);
        const size_t lvl = (size_t)(level - 1) * 2 * P.BH * (P.N / 2);
        pq = perms + lvl;
        pk = perms + lvl + (size_t)P.BH * (P.N / 2);
    }
    // at most two CTAs per SM (each holds 256 TMEM columns); persistent
    // CTAs, two per SM of a 152-SM GB300
    size_t smem = causal_attn_smem(P.d);
    if (smem < kSmemPerSM / 3 + 1024) smem = kSmemPerSM / 3 + 1024;
    const int grid = items < 2 * 152 ? items : 2 * 152;
    auto launch = [&](auto kern) {
        cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             (int)smem);
        kern<<<grid, kCaThreads, smem, st>>>(
            (const uint16_t *)q, (const uint16_t *)k, (const uint16_t *)v, pq,
            pk, P.N, n_leaf, m, P.b, items, next_item, P.scale, P.eps, RO, RL,
            status);
        return cudaGetLastError();
    };
    if (P.d == 128)
        return mode == 0 ? launch(k_causal_attn_tc<128, 0>)
                         : launch(k_causal_attn_tc<128, 1>);
    return mode == 0 ? launch(k_causal_attn_tc<64, 0>)
                     : launch(k_causal_attn_tc<64, 1>);
}

int causal_segments(const Plan &P) {
    const int nc = P.N / 128;
    int nseg = 1;
    while (nseg * 2 <= nc && nc % (nseg * 2) == 0 &&
           (long)P.BH * nseg * 2 <= 304)
        nseg *= 2;
    return nseg;
}

size_t causal_scan_smem(const Plan &P) {
    const size_t lg_pad = ((size_t)P.L * 4 + 15) / 16 * 16;
    const size_t r_pad = P.r < 128 ? 128 : P.r;
    return 1024 + (size_t)2 * 128 * P.d * 2 + 16384 +
           (lg_pad * P.d * 2 + 1023) / 1024 * 1024 + 128 * r_pad * 2;
}

cudaError_t launch_causal_scan(const Plan &P, const void *k, const void *v,
                               const uint16_t *w_bf16, float *part,
                               uint16_t *sBh, float *sA, DeviceStatus *status,
                               cudaStream_t st) {
    const int nseg = causal_segments(P);
    const int per = P.r * P.d + P.r;
    dim3 g1((per + 255) / 256, P.BH);
    k_seg_offsets<<<g1, 256, 0, st>>>(part, nseg, P.r, P.d);
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return e;
    const int G = (P.N / 128) / nseg;
    // one CTA per SM (it holds all 512 TMEM columns)
    size_t smem = causal_scan_smem(P);
    if (smem < kSmemPerSM / 2 + 1024) smem = kSmemPerSM / 2 + 1024;
    auto launch = [&](auto kern) {
        cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             (int)smem);
        kern<<<P.BH * nseg, kCaThreads, smem, st>>>(
            (const uint16_t *)k, (const uint16_t *)v, w_bf16, part, P.N, P.H,
            nseg, G, P.beta, sBh, sA, status);
        return cudaGetLastError();
    };
    if (P.d == 128) {
        if (P.L == 16) return launch(k_causal_scan<128, 16>);
        if (P.L == 8) return launch(k_causal_scan<128, 8>);
        return launch(k_causal_scan<128, 4>);
    }
    if (P.L == 16) return launch(k_causal_scan<64, 16>);
    if (P.L == 8) return launch(k_causal_scan<64, 8>);
    return launch(k_causal_scan<64, 4>);
}

cudaError_t launch_causal_race(const Plan &P, const void *q, const void *k,
                               const void *v, const uint16_t *w_bf16,
                               const uint16_t *sBh, const float *sA,
                               const float *RO, const float *RL,
                               const float *lambda_tok, const float *gates,
                               void *o, float *log_ds, float *dlr, float *m,
                               DeviceStatus *status, cudaStream_t st) {
    const int blocks = P.BH * (P.N / 128);
    // one CTA per SM (it holds all 512 TMEM columns)
    size_t smem = causal_race_smem(P);
    if (smem < kSmemPerSM / 2 + 1024) smem = kSmemPerSM / 2 + 1024;
    auto launch = [&](auto kern) {
        cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             (int)smem);
        kern<<<blocks, kCaThreads, smem, st>>>(
            (const uint16_t *)q, (const uint16_t *)k, (const uint16_t *)v,
            w_bf16, sBh, sA, RO, RL, lambda_tok, gates, P.N, P.H, P.beta,
            P.eps, P.lambda, P.fusion_mode, P.o32 ? nullptr : (uint16_t *)o,
            P.o32 ? (float *)o : nullptr, log_ds, dlr, m, status);
        return cudaGetLastError();
    };
    if (P.d == 128) {
        if (P.L == 16) return launch(k_causal_race_tc<128, 16>);
        if (P.L == 8) return launch(k_causal_race_tc<128, 8>);
        return launch(k_causal_race_tc<128, 4>);
    }
    if (P.L == 16) return launch(k_causal_race_tc<64, 16>);
    if (P.L == 8) return launch(k_causal_race_tc<64, 8>);
    return launch(k_causal_race_tc<64, 4>);
}

}  // namespace elsaa
