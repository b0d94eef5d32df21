// Persistent, warp-specialised sortLSH block attention + RACE readout +
// fusion (Algorithm "sortLSH Sparse Exact Attention Branch" block step,
// Algorithm "RACE Low-Rank Attention Branch" steps 9-10, Eq. (5)-(6)) for
// bf16 inputs whose key blocks fit one 128-key tile (b <= 128).
//
// One CTA per SM walks a contiguous range of 128-query tiles (ordered by
// head, then sorted position, so the per-head B summary, A summary and RACE
// planes are loaded once per head). Roles:
//   warp 0      loader: cp.async gathers of the tile's Q and K rows (one
//               buffer), V rows (two buffers), and per head the RACE planes
//               (as bf16), the bf16 B summary and the fp32 A summary.
//   warp 1      allocates tensor memory and issues every MMA (lane 0).
//   warps 2-9,  compute for TMEM slot 0 / slot 1 (256 columns each: scores,
//   10-17       P and pre-scaled features, then the output accumulator);
//               slot g takes the tiles of local index = g (mod 2), so one
//               slot's softmax overlaps the other slot's MMAs and loads.
//               Within a slot, warps w and w + 4 share TMEM lanes (lane
//               group w mod 4) and split each row's key columns, RACE
//               tables and output columns.

// Per tile: proj + S MMAs -> (group) features, Den, softmax, P and the
// pre-scaled features into TMEM -> PV and Phi'B MMAs into one accumulator
// -> (group) epilogue O = c1 * acc. Every hand-off is an mbarrier; every wait
// is bounded and a stalled pipeline drains through a shared abort flag.
#include "device_common.cuh"
#include "tc_common.cuh"
#include "tc_race.cuh"

namespace elsaa {

namespace {

using namespace tc;

constexpr int kWsThreads = 576;   // loader, MMA and 16 compute warps
constexpr int kWsLoaders = 32;    // warp 0
constexpr int kWsNK = 128;        // keys per query tile
// TMEM slot layout (256 columns): S/P/features region [0, 128) in four
// 32-column quarters, output accumulator [128, 128 + d). P of keys
// [64h, 64h + 64) (row half h) lives in quarter 2h, packed in place over
// the scores already read; the pre-scaled RACE features of buckets
// [0, 128) go to quarters 1 and 3, buckets [128, 256) to quarters 0 and 2
// once the P V product is done.
__device__ __forceinline__ uint32_t quarter_col(int k, int col0) {
    // K-step k (16 keys or buckets = 8 columns) of a quarter pair
    return (uint32_t)(col0 + (k < 4 ? 8 * k : 64 + 8 * (k - 4)));
}

struct WsBars {
    uint64_t qk_full, qk_empty, wb_full, head_done;
    uint64_t v_full[2], v_empty[2];
    uint64_t s_full[2], p_full[2], pv_done[2], p2_full[2], o_full[2];
    uint64_t tmem_empty[2];
};

template <int G>
__global__ void __launch_bounds__(kWsThreads, 1)
    k_block_attn_ws(const uint16_t *__restrict__ qx,
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
                    float lambda, int mode, int tiles_per_head,
                    long total_tiles, DeviceStatus *status) {
    constexpr int R = 1 << G;
    constexpr int nk = kWsNK;
    extern __shared__ unsigned char smem_raw[];
    __shared__ WsBars bars;
    __shared__ uint32_t tbase;
    __shared__ int abort_flag;
    __shared__ float xmax[2][2][128], xsum[2][2][128], xden[2][2][128];
    volatile int *abort = &abort_flag;
    const int tid = threadIdx.x, warp = tid >> 5, lane_id = tid & 31;
    const int Lg = L * G, r = L * R;
    const long t_begin = total_tiles * blockIdx.x / gridDim.x;
    const long t_end = total_tiles * (blockIdx.x + 1) / gridDim.x;
    const int ntiles = (int)(t_end - t_begin);

    const uint32_t tileB = (uint32_t)nk * d * 2u;  // one [128 x d] tile
    const uint32_t base = align1k(smem_u32(smem_raw));
    const uint32_t sQ = base;
    const uint32_t sK = sQ + tileB;
    const uint32_t sW = sK + tileB;
    const uint32_t sV0 = sW + align1k(Lg_pad * d * 2);
    const uint32_t sB = sV0 + 2 * tileB;
    const uint32_t sA = sB + align1k(r * d * 2);  // fp32 [r]
    const float *Asm = reinterpret_cast<const float *>(smem_raw + (sA - smem_u32(smem_raw)));

    if (warp == 1) tmem_alloc(&tbase, 512);
    if (tid == 0) {
        mbar_init(&bars.qk_full, kWsLoaders);
        mbar_init(&bars.qk_empty, 1);
        mbar_init(&bars.wb_full, kWsLoaders);
        mbar_init(&bars.head_done, 1);
        for (int s = 0; s < 2; ++s) {
            mbar_init(&bars.v_full[s], kWsLoaders);
            mbar_init(&bars.v_empty[s], 1);
            mbar_init(&bars.s_full[s], 1);
            mbar_init(&bars.p_full[s], 256);
            mbar_init(&bars.pv_done[s], 1);
            mbar_init(&bars.p2_full[s], 256);
            mbar_init(&bars.o_full[s], 1);
            mbar_init(&bars.tmem_empty[s], 256);
        }
        abort_flag = 0;
        fence_mbar_init();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tm = tbase;

    auto tile_head = [=](int i) {
        return (int)((t_begin + i) / tiles_per_head);
    };
    auto tile_p0 = [=](int i) {
        return (int)((t_begin + i) % tiles_per_head) * 128;
    };
    auto new_head = [=](int i) {
        return i == 0 || tile_head(i) != tile_head(i - 1);
    };
    auto head_last = [=](int i) {
        return i == ntiles - 1 || tile_head(i + 1) != tile_head(i);
    };
    auto key_pos0 = [=](int p0) { return b >= 128 ? (p0 / b) * b : p0; };

    if (warp == 0) {
        // ------------------------------------------------------------- loader
        const int lt = lane_id;
        const int chunks = d >> 3;
        constexpr int kRows = kWsNK / kWsLoaders;  // rows per loader thread
        int hc = 0;           // heads loaded
        int pending_v = -1;   // tile whose V copies are not yet signalled
        // signal_v: the V copies of tile pending_v have landed (all but the
        // newest copy group when keep_newest) -> arrive on its barrier
#define ELSAA_SIGNAL_V(keep_newest)                       \
    do {                                                  \
        if (pending_v >= 0) {                             \
            if (keep_newest)                              \
                cp_async_wait<1>();                       \
            else                                          \
                cp_async_wait<0>();                       \
            fence_proxy_async_smem();                     \
            mbar_arrive(&bars.v_full[pending_v & 1]);     \
            pending_v = -1;                               \
        }                                                 \
    } while (0)
        auto clampi = [=](int i) { return (i < 0 || i >= N) ? 0 : i; };
        auto copy_row = [=](uint32_t dst, int row, const uint16_t *g) {
            for (int c = 0; c < chunks; ++c)
                cp_async16(dst + panel_offset(row, c, nk), g + c * 8);
        };
        for (int i = 0; i < ntiles; ++i) {
            const int bh = tile_head(i), p0 = tile_p0(i), kp0 = key_pos0(p0);
            const int32_t *pq = perm_q + (size_t)bh * N;
            const int32_t *pk = perm_k + (size_t)bh * N;
            // row indices first (independent loads in flight together)
            int iq[kRows], ik[kRows];
#pragma unroll
            for (int u = 0; u < kRows; ++u) {
                iq[u] = pq[min(p0 + lt + u * kWsLoaders, N - 1)];
                ik[u] = pk[min(kp0 + lt + u * kWsLoaders, N - 1)];
            }
            const uint16_t *qh = qx + (size_t)bh * N * d;
            const uint16_t *kh = kx + (size_t)bh * N * d;
            const uint16_t *vh = vx + (size_t)bh * N * d;
            if (new_head(i)) {
                ELSAA_SIGNAL_V(false);
                if (i > 0 && !mbar_wait_or_abort(&bars.head_done, (hc - 1) & 1,
                                                 abort, status, 31))
                    break;
                load_planes_bf16(sW, w_race + (size_t)(bh % H) * Lg * d, Lg,
                                 Lg_pad, d, lt, kWsLoaders);
                load_rows(sB, Bh + (size_t)bh * r * d, r, d, d, lt,
                          kWsLoaders);
                for (int c = lt; c < r / 4; c += kWsLoaders)
                    cp_async16(sA + 16 * c, Ag + (size_t)bh * r + 4 * c);
                cp_async_commit();
                cp_async_wait<0>();
                fence_proxy_async_smem();
                mbar_arrive(&bars.wb_full);
                ++hc;
            }
            if (i > 0 && !mbar_wait_or_abort(&bars.qk_empty, (i - 1) & 1,
                                             abort, status, 32))
                break;
#pragma unroll
            for (int u = 0; u < kRows; ++u) {
                copy_row(sQ, lt + u * kWsLoaders, qh + (size_t)clampi(iq[u]) * d);
                copy_row(sK, lt + u * kWsLoaders, kh + (size_t)clampi(ik[u]) * d);
            }
            cp_async_commit();
            ELSAA_SIGNAL_V(true);
            if (i >= 2 && !mbar_wait_or_abort(&bars.v_empty[i & 1],
                                              ((i >> 1) - 1) & 1, abort,
                                              status, 33))
                break;
            const uint32_t sV = sV0 + (i & 1) * tileB;
#pragma unroll
            for (int u = 0; u < kRows; ++u)
                copy_row(sV, lt + u * kWsLoaders, vh + (size_t)clampi(ik[u]) * d);
            cp_async_commit();
            pending_v = i;
            cp_async_wait<1>();
            fence_proxy_async_smem();
            mbar_arrive(&bars.qk_full);
        }
        ELSAA_SIGNAL_V(false);
#undef ELSAA_SIGNAL_V
        cp_async_wait<0>();
    } else if (warp == 1) {
        // ----------------------------------------------------------- MMA issue
        if (lane_id == 0 && ntiles > 0) {
            const uint32_t id_proj = idesc_bf16(128, Lg_pad, false, false);
            const uint32_t id_s = idesc_bf16(128, nk, false, false);
            const uint32_t id_o = idesc_bf16(128, d, false, true);
            const int r0 = min(r, nk);
            auto finish = [&](int j) -> bool {
                const int s = j & 1, k = j >> 1;
                const uint32_t so = tm + 256u * s;
                if (!mbar_wait_or_abort(&bars.p_full[s], k & 1, abort, status,
                                        41) ||
                    !mbar_wait_or_abort(&bars.v_full[s], k & 1, abort, status,
                                        42))
                    return false;
                tc_fence_after();
                const uint32_t sV = sV0 + s * tileB;
                for (int kk = 0; kk < nk / 16; ++kk)  // O = P V
                    mma_ts(so + nk, so + quarter_col(kk, 0),
                           smem_desc(sV + kk * 2048, (uint32_t)nk * 128, 1024),
                           id_o, kk > 0);
                for (int kk = 0; kk < r0 / 16; ++kk)  // O += Phi' B
                    mma_ts(so + nk, so + quarter_col(kk, 32),
                           smem_desc(sB + kk * 2048, (uint32_t)r * 128, 1024),
                           id_o, 1);
                mma_commit(&bars.v_empty[s]);
                if (r > nk) {
                    mma_commit(&bars.pv_done[s]);
                    if (!mbar_wait_or_abort(&bars.p2_full[s], k & 1, abort,
                                            status, 43))
                        return false;
                    tc_fence_after();
                    for (int kk = 0; kk < (r - nk) / 16; ++kk)
                        mma_ts(so + nk, so + quarter_col(kk, 0),
                               smem_desc(sB + (uint32_t)nk * 128 + kk * 2048,
                                         (uint32_t)r * 128, 1024),
                               id_o, 1);
                }
                mma_commit(&bars.o_full[s]);
                if (head_last(j)) mma_commit(&bars.head_done);
                return true;
            };
            int hc = 0;
            bool ok = true;
            for (int i = 0; i < ntiles && ok; ++i) {
                const int s = i & 1;
                const uint32_t so = tm + 256u * s;
                // at a head boundary the loaders wait for the previous
                // head's MMAs (head_done) before loading the new planes and
                // B summary: finish the previous tile first
                if (i >= 1 && new_head(i)) ok = finish(i - 1);
                if (!ok) break;
                ok = mbar_wait_or_abort(&bars.qk_full, i & 1, abort, status,
                                        44);
                if (ok && new_head(i)) {
                    ok = mbar_wait_or_abort(&bars.wb_full, hc & 1, abort,
                                            status, 45);
                    ++hc;
                }
                if (ok && i >= 2)
                    ok = mbar_wait_or_abort(&bars.tmem_empty[s],
                                            ((i >> 1) - 1) & 1, abort, status,
                                            46);
                if (!ok) break;
                tc_fence_after();
                for (int kk = 0; kk < d / 16; ++kk) {
                    uint32_t oq = (kk >> 2) * 128 * 128 + (kk & 3) * 32;
                    uint32_t ow = (kk >> 2) * Lg_pad * 128 + (kk & 3) * 32;
                    uint64_t aq = smem_desc(sQ + oq, 16, 1024);
                    mma_ss(so + nk, aq, smem_desc(sW + ow, 16, 1024), id_proj,
                           kk > 0);
                    mma_ss(so, aq, smem_desc(sK + oq, 16, 1024), id_s, kk > 0);
                }
                mma_commit(&bars.s_full[s]);
                mma_commit(&bars.qk_empty);
                if (i >= 1 && !new_head(i)) ok = finish(i - 1);
            }
            if (ok) finish(ntiles - 1);
        }
        __syncwarp();
    } else {
        // ------------------------------------------------------ compute groups
        // warps 2-9: slot 0, warps 10-17: slot 1; within a slot, warps
        // (w, w + 4) share TMEM lanes and split the row in two halves.
        const int cw = warp - 2;
        const int g = cw >> 3;                       // TMEM slot / tile parity
        const int half = (cw >> 2) & 1;
        const int row = (warp & 3) * 32 + lane_id;   // query row = TMEM lane
        const uint32_t lane = (uint32_t)((warp & 3) * 32) << 16;
        const int split = table_split(L, G);
        const int l0 = half ? split : 0, l1 = half ? L : split;
        const float sl2e = scale * kLog2e;
        const int r0 = min(r, nk);
        const int kbeg = half * (nk / 2);
        auto wwait = [=](uint64_t *bar, uint32_t par, int site) {
            return __all_sync(0xffffffffu,
                              mbar_wait_or_abort(bar, par, abort, status,
                                                 site));
        };
        for (int j = g; j < ntiles; j += 2) {
            const int k = j >> 1;
            const uint32_t so = tm + 256u * g + lane;
            const int bh = tile_head(j), p0 = tile_p0(j);
            const int qpos = p0 + row;
            const bool qvalid = qpos < N;
            int qi = perm_q[(size_t)bh * N + min(qpos, N - 1)];  // prefetch
            if (!wwait(&bars.s_full[g], k & 1, 51)) break;
            tc_fence_after();
            // RACE features of this half's tables and partial Den (A from
            // shared memory: the loaders stage it with the planes; the MMA
            // warp only starts tile j after that head's stage completed)
            float sp[32];
            race_bits32(so + nk + l0 * G, (l1 - l0) * G, beta, sp);
            float dacc[4] = {0.0f, 0.0f, 0.0f, 0.0f};  // independent chains
#pragma unroll
            for (int lt = 0; lt < 32 / G; ++lt) {
                if (G == 4 && l0 + lt < l1) {
                    float u[4], w[4];
                    table_uw4(&sp[lt * G], 1.0f, u, w);
                    dacc[lt & 3] += table_dot4(u, w, Asm + (l0 + lt) * R);
                } else if (l0 + lt < l1) {
                    float phi[R];
                    table_phi<G>(&sp[lt * G], phi);
                    const float *a = Asm + (l0 + lt) * R;
                    if (R >= 4) {
#pragma unroll
                        for (int q = 0; q < R; q += 4) {
                            const float4 a4 =
                                *reinterpret_cast<const float4 *>(a + q);
                            dacc[0] = fmaf(phi[q], a4.x, dacc[0]);
                            dacc[1] = fmaf(phi[q + 1], a4.y, dacc[1]);
                            dacc[2] = fmaf(phi[q + 2], a4.z, dacc[2]);
                            dacc[3] = fmaf(phi[q + 3], a4.w, dacc[3]);
                        }
                    } else {
#pragma unroll
                        for (int q = 0; q < R; ++q)
                            dacc[q & 3] = fmaf(phi[q], a[q], dacc[q & 3]);
                    }
                }
            }
            const float den = (dacc[0] + dacc[1]) + (dacc[2] + dacc[3]);
            // softmax over this half's key columns
            const int klo = b < 128 ? (row / b) * b : 0;
            const int khi = b < 128 ? klo + b : nk;
            float mxa[4] = {-INFINITY, -INFINITY, -INFINITY, -INFINITY};
            const bool masked = b < 128;
#pragma unroll
            for (int c = 0; c < nk / 2; c += 32) {
                uint32_t v0[16], v1[16];
                tmem_ld16(so + kbeg + c, v0);
                tmem_ld16(so + kbeg + c + 16, v1);
                tmem_wait_ld();
                if (!masked) {
#pragma unroll
                    for (int jj = 0; jj < 16; ++jj)
                        mxa[jj & 3] = fmaxf(mxa[jj & 3],
                                            fmaxf(__uint_as_float(v0[jj]),
                                                  __uint_as_float(v1[jj])));
                } else {
#pragma unroll
                    for (int jj = 0; jj < 16; ++jj) {
                        const int key0 = kbeg + c + jj, key1 = key0 + 16;
                        if (key0 >= klo && key0 < khi)
                            mxa[jj & 3] =
                                fmaxf(mxa[jj & 3], __uint_as_float(v0[jj]));
                        if (key1 >= klo && key1 < khi)
                            mxa[jj & 3] =
                                fmaxf(mxa[jj & 3], __uint_as_float(v1[jj]));
                    }
                }
            }
            float mx = fmaxf(fmaxf(mxa[0], mxa[1]), fmaxf(mxa[2], mxa[3]));
            xmax[g][half][row] = mx;
            xden[g][half][row] = den;
            named_sync(1 + g, 256);
            mx = fmaxf(xmax[g][0][row], xmax[g][1][row]);
            const float denf =
                (xden[g][0][row] + xden[g][1][row]) * (1.0f / (float)L);
            const float M2 = mx * sl2e;
            float ls[4] = {0.0f, 0.0f, 0.0f, 0.0f};
#pragma unroll
            for (int c = 0; c < nk / 2; c += 32) {
                uint32_t v[2][16];
                tmem_ld16(so + kbeg + c, v[0]);
                tmem_ld16(so + kbeg + c + 16, v[1]);
                tmem_wait_ld();
                uint32_t pk16[16];
#pragma unroll
                for (int hh = 0; hh < 2; ++hh) {
#pragma unroll
                    for (int jj = 0; jj < 16; jj += 2) {
                        const int key = kbeg + c + 16 * hh + jj;
                        float a0 = ex2_approx(
                            fmaf(__uint_as_float(v[hh][jj]), sl2e, -M2));
                        float a1 = ex2_approx(
                            fmaf(__uint_as_float(v[hh][jj + 1]), sl2e, -M2));
                        if (masked) {
                            a0 = (key >= klo && key < khi) ? a0 : 0.0f;
                            a1 = (key + 1 >= klo && key + 1 < khi) ? a1 : 0.0f;
                        }
                        ls[(jj >> 1) & 3] += a0 + a1;
                        pk16[8 * hh + (jj >> 1)] = pack_bf16x2(a0, a1);
                    }
                }
                // quarter 2h, over scores of this half already read
                tmem_st16(so + kbeg + (c >> 1), pk16);
            }
            float lsum = (ls[0] + ls[1]) + (ls[2] + ls[3]);
            xsum[g][half][row] = lsum;
            tc_fence_before();
            named_sync(1 + g, 256);  // every S read of the slot is done
            tc_fence_after();
            lsum = xsum[g][0][row] + xsum[g][1][row];
            // fusion scalars (Eq. (5) in log-sum-exp form, Eq. (6))
            qi = (qi < 0 || qi >= N) ? 0 : qi;
            const size_t tok = (size_t)bh * N + qi;
            const float log_ds = M2 * kLn2 + __logf(lsum);
            const float lam = (lambda_tok && qvalid) ? lambda_tok[tok] : lambda;
            const float gs = (gates && qvalid) ? gates[2 * tok] : 1.0f;
            const float gl = (gates && qvalid) ? gates[2 * tok + 1] : 1.0f;
            const float msp =
                fusion_multiplier_fast(log_ds, lam, denf, eps, mode);
            const float c1 =
                __fdividef(gs * msp, lsum + eps * ex2_approx(-M2));
            const float c1e = fmaxf(c1, 1e-30f);
            const float ratio =
                __fdividef(gl, (float)L * (denf + eps) * c1e);
            const int b0 = l0 * R, b1 = l1 * R;  // this half's buckets
            if (b0 < r0 && b1 > b0)
                write_phi_tmem_q<G>(sp, l0, l1, r, ratio, 0, r0, so + 32);
            tmem_wait_st();
            tc_fence_before();
            mbar_arrive(&bars.p_full[g]);
            if (r > nk) {
                if (!wwait(&bars.pv_done[g], k & 1, 52)) break;
                tc_fence_after();
                if (b1 > nk && b1 > b0)
                    write_phi_tmem_q<G>(sp, l0, l1, r, ratio, nk, r, so);
                tmem_wait_st();
                tc_fence_before();
                mbar_arrive(&bars.p2_full[g]);
            }
            if (!wwait(&bars.o_full[g], k & 1, 53)) break;
            tc_fence_after();
            uint16_t *orow = ox + tok * d;
            for (int c = half * (d >> 1); c < (half + 1) * (d >> 1); c += 32) {
                uint32_t v[32];
                tmem_ld16(so + nk + c, *reinterpret_cast<uint32_t(*)[16]>(&v[0]));
                tmem_ld16(so + nk + c + 16,
                          *reinterpret_cast<uint32_t(*)[16]>(&v[16]));
                tmem_wait_ld();
                if (qvalid) {
                    uint4 *dst = reinterpret_cast<uint4 *>(orow + c);
#pragma unroll
                    for (int q = 0; q < 4; ++q) {
                        uint4 w;
                        w.x = pack_bf16x2(c1e * __uint_as_float(v[8 * q]),
                                          c1e * __uint_as_float(v[8 * q + 1]));
                        w.y = pack_bf16x2(c1e * __uint_as_float(v[8 * q + 2]),
                                          c1e * __uint_as_float(v[8 * q + 3]));
                        w.z = pack_bf16x2(c1e * __uint_as_float(v[8 * q + 4]),
                                          c1e * __uint_as_float(v[8 * q + 5]));
                        w.w = pack_bf16x2(c1e * __uint_as_float(v[8 * q + 6]),
                                          c1e * __uint_as_float(v[8 * q + 7]));
                        dst[q] = w;
                    }
                }
            }
            if (qvalid && half == 0) {
                if (log_ds_out) log_ds_out[tok] = log_ds;
                if (dlr_out) dlr_out[tok] = denf;
                if (m_out) m_out[tok] = msp;
            }
            tc_fence_before();
            mbar_arrive(&bars.tmem_empty[g]);
        }
    }
    tc_fence_before();
    __syncthreads();
    if (warp == 1) tmem_dealloc(tm, 512);
}

}  // namespace

bool ws_supported(const Plan &P) {
    return tc_supported(P) && P.b <= 128;
}

cudaError_t launch_block_attn_ws(
    const Plan &P, const void *q, const void *k, const void *v,
    const float *w_race, const int32_t *perm_q, const int32_t *perm_k,
    const float *A, const uint16_t *Bh, const float *lambda_tok,
    const float *gates, void *o, float *log_d_sparse, float *d_lr,
    float *m_sparse, DeviceStatus *status, cudaStream_t st) {
    const int lg_pad = (P.L * P.gamma + 15) / 16 * 16;
    const size_t tileB = (size_t)kWsNK * P.d * 2;
    const size_t smem = 1024 + 4 * tileB + ((size_t)lg_pad * P.d * 2 + 1023) /
                                               1024 * 1024 +
                        ((size_t)P.r * P.d * 2 + 1023) / 1024 * 1024 +
                        (size_t)P.r * 4;
    const int tiles_per_head = (P.N + 127) / 128;
    const long total = (long)tiles_per_head * P.BH;
    int dev = 0, sms = 148;
    if (cudaGetDevice(&dev) == cudaSuccess)
        cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    const int grid = (int)(total < sms ? total : sms);
    const int lg = lg_pad;
    auto launch = [&](auto kern) {
        cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             (int)smem);
        kern<<<grid, kWsThreads, smem, st>>>(
            (const uint16_t *)q, (const uint16_t *)k, (const uint16_t *)v,
            w_race, perm_q, perm_k, A, Bh, lambda_tok, gates, (uint16_t *)o,
            log_d_sparse, d_lr, m_sparse, P.N, P.d, P.H, P.b, P.L, lg, P.beta,
            P.eps, P.scale, P.lambda, P.fusion_mode, tiles_per_head, total,
            status);
        return cudaGetLastError();
    };
    switch (P.gamma) {
        case 1: return launch(k_block_attn_ws<1>);
        case 2: return launch(k_block_attn_ws<2>);
        case 3: return launch(k_block_attn_ws<3>);
        case 4: return launch(k_block_attn_ws<4>);
        case 5: return launch(k_block_attn_ws<5>);
        case 6: return launch(k_block_attn_ws<6>);
        default: return cudaErrorInvalidValue;
    }
}

}  // namespace elsaa
