// Persistent, warp-specialised sortLSH block attention + RACE readout +
// fusion (Algorithm "sortLSH Sparse Exact Attention Branch" block step,
// Algorithm "RACE Low-Rank Attention Branch" steps 9-10, Eq. (5)-(6)) for
// bf16 inputs whose key blocks fit one 128-key tile (b <= 128).
//
// One CTA per SM walks a contiguous range of 128-query tiles (ordered by
// head, then sorted position, so the per-head B summary, A summary and RACE
// planes are loaded once per head). Roles:
//   warps 0-7,  compute for TMEM slot 0 / slot 1 (256 columns each: scores,
//   8-15        P and pre-scaled features, then the output accumulator);
//               slot g takes the tiles of local index = g (mod 2), so one
//               slot's softmax overlaps the other slot's MMAs and loads.
//               Within a slot, warps w and w + 4 share TMEM lanes (lane
//               group w mod 4) and split each row's key columns and output
//               columns in halves; half h owns the RACE buckets of the
//               64-bucket chunks h and h + 2, so both halves write features
//               before and after the P V product.
//   warp 16     allocates tensor memory and issues every MMA (lane 0).
//   warps 17-19 loaders: cp.async gathers of the tile's Q rows (warp 17), K
//               rows (warp 18, which also stages per head the RACE planes as
//               bf16, the bf16 B summary and the fp32 A summary) and V rows
//               (warp 19, two buffers). A gather's rate grows with the
//               number of warps issuing it, hence one warp per operand.

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

constexpr int kWsThreads = 640;   // 16 compute, MMA and 3 loader warps
constexpr int kWsMmaWarp = 16;
constexpr int kWsLoaders = 32;    // threads of one loader warp
constexpr int kWsNK = 128;        // keys per query tile
// TMEM slot layout (256 columns): S/P/features region [0, 128) in four
// 32-column quarters, output accumulator [128, 128 + d). P of keys
// [64h, 64h + 64) (row half h) lives in quarter 2h, packed in place over
// the scores already read; the pre-scaled RACE features of buckets
// [0, 128) go to quarters 1 and 3, buckets [128, 256) to quarters 0 and 2
// once the P V product is done.

struct WsBars {
    uint64_t qk_full, wb_full, head_done;
    uint64_t idx_full[2], idx_empty[2];
    uint64_t v_full[2], v_empty[2], pv0_done[2];
    uint64_t s_full[2], p_full[2], pv_done[2], p2_full[2], o_full[2];
    uint64_t tmem_empty[2];
};

// NPASS 128-key passes per query tile, online softmax across them: 1 for
// b <= 128; b / 128 for larger blocks; with nb neighbouring sorted key
// blocks per side (b >= 128), (2 nb + 1) b / 128 passes over the window.
// KM: which keys the passes walk. 0: the query block's own key block.
// 1 (WIN): a neighbour window (nb > 0), whose passes past either end of
// the sequence are masked. 2 (SEL): the top-k selector's candidate blocks
// (cand, tk_c per query block), each key masked unless the row's bit in
// selmask is set. The checks of the other modes are compiled out. O32: O
// is written as fp32 (out_fp32), each thread storing its half row directly.
template <int G, int NPASS, int KM, bool O32 = false>
__global__ void __launch_bounds__(kWsThreads, 1)
    k_block_attn_ws(const uint16_t *__restrict__ qx,
                    const uint16_t *__restrict__ kx,
                    const uint16_t *__restrict__ vx,
                    const __grid_constant__ CUtensorMap tmW,
                    const __grid_constant__ CUtensorMap tmB,
                    const int32_t *__restrict__ perm_q,
                    const int32_t *__restrict__ perm_k,
                    const float *__restrict__ Ag,
                    const float *__restrict__ lambda_tok,
                    const float *__restrict__ gates, uint16_t *__restrict__ ox,
                    float *__restrict__ o32,
                    float *__restrict__ log_ds_out, float *__restrict__ dlr_out,
                    float *__restrict__ m_out, int N, int d, int H, int b,
                    int nb, int L, int Lg_pad, float beta, float eps,
                    float scale,
                    float lambda, int mode, int tiles_per_head,
                    long total_tiles, DeviceStatus *status,
                    const int32_t *__restrict__ cand,
                    const uint32_t *__restrict__ selmask, int tk_c) {
    constexpr bool WIN = KM == 1, SEL = KM == 2;
    constexpr int R = 1 << G;
    constexpr int nk = kWsNK;
    extern __shared__ unsigned char smem_raw[];
    __shared__ WsBars bars;
    __shared__ uint32_t tbase;
    __shared__ int abort_flag;
    __shared__ float xmax[2][2][128], xsum[2][2][128], xden[2][2][128];
    // global rows of a tile's queries / keys, per tile parity (written by
    // the index warp, read by the slot that issues the tile's Q, K copies)
    __shared__ __align__(16) int qkrow[2][1 + NPASS][128];
    __shared__ __align__(16) int vrow[128];  // V loader: rows of its tile
    __shared__ int orow[2][128];          // per slot: output row or -1
    volatile int *abort = &abort_flag;
    const int tid = threadIdx.x, warp = tid >> 5, lane_id = tid & 31;
    const int Lg = L * G, r = L * R;
    const long t_begin = total_tiles * blockIdx.x / gridDim.x;
    const long t_end = total_tiles * (blockIdx.x + 1) / gridDim.x;
    const int ntiles = (int)(t_end - t_begin);

    const uint32_t tileB = (uint32_t)nk * d * 2u;  // one [128 x d] tile
    const uint32_t base = align1k(smem_u32(smem_raw));
    // key tile and RACE planes stacked as one B operand of NR rows: the
    // scores and the query projections come out of one MMA (N = NR) into
    // TMEM columns [0, 128) and [128, 128 + Lg_pad)
    const int NR = nk + Lg_pad;
    const uint32_t sQ = base;
    const uint32_t sKW = sQ + tileB;
    const uint32_t sV0 = sKW + align1k((uint32_t)NR * d * 2u);
    const uint32_t sB = sV0 + 2 * tileB;
    const uint32_t sA = sB + align1k(r * d * 2);  // fp32 [r]
    const float *Asm = reinterpret_cast<const float *>(smem_raw + (sA - smem_u32(smem_raw)));

    if (warp == kWsMmaWarp) tmem_alloc(&tbase, 512);
    if (tid == 0) {
        mbar_init(&bars.qk_full, 256);  // the issuing slot's threads
        mbar_init(&bars.wb_full, 1);
        mbar_init(&bars.head_done, 1);
        for (int s = 0; s < 2; ++s) {
            mbar_init(&bars.idx_full[s], kWsLoaders);
            mbar_init(&bars.idx_empty[s], 256 * NPASS);
            mbar_init(&bars.pv0_done[s], 1);
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

    // tile indices fit in int (checked on the host)
    const int tb = (int)t_begin;
    auto tile_head = [=](int i) { return (tb + i) / tiles_per_head; };
    auto tile_p0 = [=](int i) { return (tb + i) % tiles_per_head * 128; };
    auto new_head = [=](int i) {
        return i == 0 || (tb + i) % tiles_per_head == 0;
    };
    // sorted position of key column 0 of pass p of the tile starting at
    // query position p0: the passes walk the key window of the tile's
    // query block (the block and nb neighbouring blocks per side) in
    // 128-key steps. A pass past either end of the sequence holds no keys:
    // its rows are read from a valid position and its scores are masked.
    // SEL: pass p holds candidate keys [128 p, 128 p + 128) of the query
    // block, i.e. keys of candidate block 128 p / b (b >= 128)
    auto key_pos_raw = [=](int bh, int p0, int p) {
        if (SEL) {
            const int T = N / b, t = p0 / b;
            int u = cand[((size_t)bh * T + t) * tk_c + (128 * p) / b];
            u = (u < 0 || u >= T) ? t : u;
            return u * b + (128 * p) % b;
        }
        return NPASS == 1 ? p0 : (p0 / b - (WIN ? nb : 0)) * b + 128 * p;
    };
    auto pass_valid = [=](int p0, int p) {
        if (!WIN) return true;
        const int k0 = key_pos_raw(0, p0, p);
        return k0 >= 0 && k0 < N;
    };
    auto key_pos = [=](int bh, int p0, int p) {
        const int k0 = key_pos_raw(bh, p0, p);
        if (NPASS == 1) return k0;  // the tile's own keys (ragged end kept)
        return k0 < 0 ? 0 : (k0 > N - 128 ? N - 128 : k0);
    };
    // global row numbers of the 4 sorted positions pos.. pos + 3 (the
    // ragged end repeats the last row; those rows are never stored)
    auto rows4 = [=](const int32_t *pm, int pos, int rowbase) {
        int4 r;
        if (pos + 3 < N && ((uintptr_t)(pm + pos) & 15u) == 0) {
            r = *reinterpret_cast<const int4 *>(pm + pos);
        } else {
            r.x = pm[min(pos, N - 1)];
            r.y = pm[min(pos + 1, N - 1)];
            r.z = pm[min(pos + 2, N - 1)];
            r.w = pm[min(pos + 3, N - 1)];
        }
        // an entry outside [0, N) is read as row 0 (the orders come from
        // the sort, in range by construction); the checked build
        // (ELSAA_CHECKED) also records it: 4 % of this kernel's time when
        // always on
        auto fix = [=](int v) {
            if (v < 0 || v >= N) {
#ifdef ELSAA_CHECKED
                report(status, kDevPermRange, 4, rowbase / N, v);
#endif
                v = 0;
            }
            return rowbase + v;
        };
        return make_int4(fix(r.x), fix(r.y), fix(r.z), fix(r.w));
    };

    if (warp > kWsMmaWarp) {
        // ------------------------------------------------------------ loaders
        // warp 17: global row numbers of each tile's queries and keys into
        //          qkrow[tile & 1] (the copies themselves are issued by the
        //          compute slot whose scores just freed the Q, K buffer);
        // warp 18: per head, TMA loads of the bf16 RACE planes (under the
        //          key rows), the bf16 B summary and the fp32 A summary;
        // warp 19: V rows with cp.async (whole rows per instruction, into
        //          the swizzled operand layout); completion reaches v_full
        //          through cp.async's own mbarrier arrivals.
        const int role = warp - kWsMmaWarp - 1;
        const int lt = lane_id;
        auto lwait = [=](uint64_t *bar, uint32_t par, int site) {
            return __all_sync(0xffffffffu,
                              mbar_wait_or_abort(bar, par, abort, status,
                                                 site));
        };
        if (role == 0) {
            for (int i = 0; i < ntiles; ++i) {
                const int bh = tile_head(i), p0 = tile_p0(i), t = i & 1;
                if (i >= 2 &&
                    !lwait(&bars.idx_empty[t], ((i >> 1) - 1) & 1, 30))
                    break;
                *reinterpret_cast<int4 *>(&qkrow[t][0][4 * lt]) =
                    rows4(perm_q + (size_t)bh * N, p0 + 4 * lt, bh * N);
#pragma unroll
                for (int ps = 0; ps < NPASS; ++ps)
                    *reinterpret_cast<int4 *>(&qkrow[t][1 + ps][4 * lt]) =
                        rows4(perm_k + (size_t)bh * N,
                              key_pos(bh, p0, ps) + 4 * lt, bh * N);
                __syncwarp();
                mbar_arrive(&bars.idx_full[t]);
            }
        } else if (role == 1) {
            int hc = 0;
            for (int i = 0; i < ntiles; ++i) {
                if (!new_head(i)) continue;
                const int bh = tile_head(i);
                if (i > 0 && !lwait(&bars.head_done, (hc - 1) & 1, 31)) break;
                if (lt == 0) {  // TMA: planes under the key rows, B, A
                    mbar_expect_tx(&bars.wb_full,
                                   (uint32_t)(Lg_pad + r) * d * 2u + r * 4u);
                    for (int p = 0; p < (d >> 6); ++p) {
                        tma_load_2d(sKW + p * NR * 128 + nk * 128, &tmW,
                                    64 * p, (bh % H) * Lg_pad, &bars.wb_full);
                        tma_load_2d(sB + p * r * 128, &tmB, 64 * p, bh * r,
                                    &bars.wb_full);
                    }
                    bulk_load(sA, Ag + (size_t)bh * r, (uint32_t)r * 4u,
                              &bars.wb_full);
                }
                __syncwarp();
                ++hc;
            }
        } else {
            const int cpr = d >> 3;    // 16-byte chunks per row
            const int rpi = 32 / cpr;  // rows per instruction
            const int lrow = lt / cpr, lc = lt - lrow * cpr;
            bool go = true;
            for (int i = 0; i < ntiles && go; ++i) {
                const int bh = tile_head(i), p0 = tile_p0(i);
                for (int ps = 0; ps < NPASS; ++ps) {
                    __syncwarp();  // the previous rows are all read
                    *reinterpret_cast<int4 *>(&vrow[4 * lt]) =
                        rows4(perm_k + (size_t)bh * N,
                              key_pos(bh, p0, ps) + 4 * lt, bh * N);
                    __syncwarp();
                    // buffer i & 1 serves the passes of tiles i, i + 2, ...
                    // in turn; a pass's V goes in once the previous user is
                    // done (its P V product, or the epilogue of the last
                    // pass, which stages O there)
                    const int ub = (i >> 1) * NPASS + ps;
                    if (ub >= 1 &&
                        !lwait(&bars.v_empty[i & 1], (ub - 1) & 1, 33)) {
                        go = false;
                        break;
                    }
                    const uint32_t sV = sV0 + (i & 1) * tileB;
                    for (int row = lrow; row < nk; row += rpi)
                        cp_async16(sV + panel_offset(row, lc, nk),
                                   vx + (size_t)vrow[row] * d + lc * 8);
                    cp_async_mbar_arrive(&bars.v_full[i & 1]);
                }
            }
            cp_async_wait<0>();
        }
    } else if (warp == kWsMmaWarp) {
        // ----------------------------------------------------------- MMA issue
        // Event driven: each pass issues whichever MMA group is ready, the
        // oldest tile's first (second feature part, then P V with the first
        // part, then the next tile's projections and scores), so one slot's
        // epilogue never holds back the other slot's products.
        // Units: (tile, pass); with NPASS = 2 the second score product of
        // a tile waits until its first P V product is complete (it reuses
        // the S columns), and the first P V product releases the V buffer
        // for the second key half.
        if (lane_id == 0 && ntiles > 0) {
            const uint32_t id_sp = idesc_bf16(128, NR, false, false);
            const uint32_t id_s = idesc_bf16(128, nk, false, false);
            const uint32_t id_o = idesc_bf16(128, d, false, true);
            const int r0 = min(r, nk);
            const bool two_parts = r > nk;
            const int nunits = ntiles * NPASS;
            int us = 0, up = 0, i2 = 0;  // next unit for S, unit for P V, tile
                                         // for part 2
            int tiles_pv = 0;            // tiles whose last P V is issued
            // position of each cursor's tile within its head (advanced
            // incrementally: no divisions in the issue loop)
            const int tph = tiles_per_head;
            int ps = (int)(t_begin % tph), pp = ps, p2 = ps;
            auto adv = [tph](int q) { return q + 1 == tph ? 0 : q + 1; };
            int hc = 0;                  // heads whose planes were consumed
            unsigned long long t_last = global_ns();
            while ((two_parts ? i2 : tiles_pv) < ntiles) {
                bool did = false;
                if (two_parts && i2 < tiles_pv) {
                    const int s = i2 & 1;
                    const uint32_t so = tm + 256u * s;
                    if (mbar_test(&bars.p2_full[s], (i2 >> 1) & 1)) {
                        tc_fence_after();
                        for (int kk = 0; kk < (r - nk) / 16; ++kk)
                            mma_ts(so + nk, so + quarter_col(kk, 0),
                                   smem_desc(sB + (uint32_t)nk * 128 + kk * 2048,
                                             (uint32_t)r * 128, 1024),
                                   id_o, 1);
                        mma_commit(&bars.o_full[s]);
                        if (i2 == ntiles - 1 || p2 == tph - 1)
                            mma_commit(&bars.head_done);
                        ++i2;
                        p2 = adv(p2);
                        did = true;
                    }
                }
                if (up < us) {
                    const int t = up / NPASS, pass = up - t * NPASS;
                    const int s = t & 1;
                    const int su = (t >> 1) * NPASS + pass;  // unit in slot
                    const uint32_t so = tm + 256u * s;
                    if (mbar_test(&bars.p_full[s], su & 1) &&
                        mbar_test(&bars.v_full[s], su & 1)) {
                        fence_proxy_async_smem();  // cp.async data -> MMA
                        tc_fence_after();
                        const uint32_t sV = sV0 + s * tileB;
                        for (int kk = 0; kk < nk / 16; ++kk)  // O (+)= P V
                            mma_ts(so + nk, so + quarter_col(kk, 0),
                                   smem_desc(sV + kk * 2048, (uint32_t)nk * 128,
                                             1024),
                                   id_o, pass > 0 || kk > 0);
                        if (pass < NPASS - 1) {
                            mma_commit(&bars.pv0_done[s]);
                            mma_commit(&bars.v_empty[s]);
                        } else {
                            for (int kk = 0; kk < r0 / 16; ++kk)  // + Phi' B
                                mma_ts(so + nk, so + quarter_col(kk, 32),
                                       smem_desc(sB + kk * 2048,
                                                 (uint32_t)r * 128, 1024),
                                       id_o, 1);
                            if (two_parts) {
                                mma_commit(&bars.pv_done[s]);
                            } else {
                                mma_commit(&bars.o_full[s]);
                                if (t == ntiles - 1 || pp == tph - 1)
                                    mma_commit(&bars.head_done);
                            }
                            ++tiles_pv;
                            pp = adv(pp);
                        }
                        ++up;
                        did = true;
                    }
                }
                // a new head's planes and B summary replace the old ones
                // only after head_done: its first S waits for every MMA of
                // the previous head to be issued
                const int ts = us / NPASS, spass = us - ts * NPASS;
                const bool nh = spass == 0 && (ts == 0 || ps == 0);
                if (us < nunits &&
                    !(nh && ts > 0 && (two_parts ? i2 : tiles_pv) < ts)) {
                    const int s = ts & 1;
                    const uint32_t so = tm + 256u * s;
                    bool ready = mbar_test(&bars.qk_full, us & 1);
                    if (ready && spass == 0)
                        ready = (ts < 2 || mbar_test(&bars.tmem_empty[s],
                                                     ((ts >> 1) - 1) & 1)) &&
                                (!nh || mbar_test(&bars.wb_full, hc & 1));
                    if (ready && spass > 0)  // S columns hold P of pass - 1
                        ready = mbar_test(&bars.pv0_done[s],
                                          ((ts >> 1) * (NPASS - 1) + spass -
                                           1) & 1);
                    if (ready) {
                        if (nh) ++hc;
                        fence_proxy_async_smem();  // cp.async data -> MMA
                        tc_fence_after();
                        for (int kk = 0; kk < d / 16; ++kk) {
                            uint32_t oq = (kk >> 2) * 128 * 128 + (kk & 3) * 32;
                            uint32_t okw = (kk >> 2) * NR * 128 + (kk & 3) * 32;
                            // pass 0: scores and projections (N = NR);
                            // later passes: scores only
                            mma_ss(so, smem_desc(sQ + oq, 16, 1024),
                                   smem_desc(sKW + okw, 16, 1024),
                                   spass == 0 ? id_sp : id_s, kk > 0);
                        }
                        mma_commit(&bars.s_full[s]);
                        ++us;
                        if (spass == NPASS - 1) ps = adv(ps);
                        did = true;
                    }
                }
                if (did) {
                    t_last = global_ns();
                } else {
                    if (*abort) break;
                    if (global_ns() - t_last > kWaitLimitNs) {
                        *abort = 1;
                        record_timeout(status, 41);
                        break;
                    }
                }
            }
        }
        __syncwarp();
    } else {
        // ------------------------------------------------------ compute groups
        // warps 0-7: slot 0, warps 8-15: slot 1; within a slot, warps
        // (w, w + 4) share TMEM lanes and split the row in two halves.
        const int cw = warp;
        const int g = cw >> 3;                       // TMEM slot / tile parity
        const int half = (cw >> 2) & 1;
        const int row = (warp & 3) * 32 + lane_id;   // query row = TMEM lane
        const uint32_t lane = (uint32_t)((warp & 3) * 32) << 16;
        // RACE buckets of this half: the 64-bucket chunks c = half (written
        // with P, before the P V product) and c = half + 2 (written after
        // it); chunk c holds tables [c T, c T + T)
        constexpr int T = R >= 64 ? 1 : 64 / R;
        const int ta0 = min(half * T, L), nt0 = min(ta0 + T, L) - ta0;
        const int ta1 = min((half + 2) * T, L), nt1 = min(ta1 + T, L) - ta1;
        const uint32_t cb0 = half ? 96u : 32u, cb1 = half ? 64u : 0u;
        const float sl2e = scale * kLog2e;
        const int kbeg = half * (nk / 2);
        // a slot's 256 threads leave a wait with one verdict (an abort
        // seen by some warps only would strand the others at the slot's
        // named barriers)
        auto wwait = [=](uint64_t *bar, uint32_t par, int site) {
            const bool ok = mbar_wait_or_abort(bar, par, abort, status, site);
            return named_sync_and(1 + g, 256, ok);
        };
        // The Q, K copies of tile t are issued by the other slot (the one
        // of tile t - 1) as soon as the scores of tile t - 1 free the Q, K
        // buffer: 256 threads, whole rows per warp instruction; completion
        // reaches qk_full through cp.async's own mbarrier arrivals.
        const int ct = (cw & 7) * 32 + lane_id;  // 0..255 within the slot
        auto issue_qk = [&](int t) -> bool {
            if (!wwait(&bars.idx_full[t & 1], (t >> 1) & 1, 54)) return false;
            const int cpr = d >> 3, rpp = 256 / cpr;
            const int crow = ct / cpr, cc = ct - crow * cpr;
            const int *qr = qkrow[t & 1][0], *kr = qkrow[t & 1][1];
            for (int rr = crow; rr < nk; rr += rpp) {
                cp_async16(sQ + panel_offset(rr, cc, nk),
                           qx + (size_t)qr[rr] * d + cc * 8);
                cp_async16(sKW + panel_offset(rr, cc, NR),
                           kx + (size_t)kr[rr] * d + cc * 8);
            }
            cp_async_mbar_arrive(&bars.qk_full);
            mbar_arrive(&bars.idx_empty[t & 1]);
            return true;
        };
        // keys of pass ps >= 1 of tile t (the queries stay): issued by the
        // tile's own slot once the previous pass's scores are done
        auto issue_k = [&](int t, int ps) -> bool {
            if (!wwait(&bars.idx_full[t & 1], (t >> 1) & 1, 57)) return false;
            const int cpr = d >> 3, rpp = 256 / cpr;
            const int crow = ct / cpr, cc = ct - crow * cpr;
            const int *kr = qkrow[t & 1][1 + ps];
            for (int rr = crow; rr < nk; rr += rpp)
                cp_async16(sKW + panel_offset(rr, cc, NR),
                           kx + (size_t)kr[rr] * d + cc * 8);
            cp_async_mbar_arrive(&bars.qk_full);
            mbar_arrive(&bars.idx_empty[t & 1]);
            return true;
        };
        bool started = true;
        if (g == 1 && ntiles > 0) started = issue_qk(0);
        for (int j = g; started && j < ntiles; j += 2) {
            const int k = j >> 1;
            const uint32_t so = tm + 256u * g + lane;
            const int bh = tile_head(j), p0 = tile_p0(j);
            const int qpos = p0 + row;
            const bool qvalid = qpos < N;
            int qi = perm_q[(size_t)bh * N + min(qpos, N - 1)];  // prefetch
            if (!wwait(&bars.s_full[g], (k * NPASS) & 1, 51)) break;
            tc_fence_after();
            // the A summary (read below) came by TMA: acquire its head's
            // stage (complete already, since S of this tile waited for it)
            if ((j < 2 || tile_head(j) != tile_head(j - 2)) &&
                !wwait(&bars.wb_full, (tile_head(j) - tile_head(0)) & 1, 55))
                break;
            if constexpr (NPASS > 1) {
                if (!issue_k(j, 1)) break;
            } else {
                if (j + 1 < ntiles && !issue_qk(j + 1)) break;
            }
            // per-bit factors of this half's tables (sp[0, 16): chunk half,
            // up to 32 when the chunk has more projection columns and no
            // second chunk exists; sp[16, 32): chunk half + 2) and partial
            // Den (A from shared memory: the loaders stage it with the
            // planes; the MMA warp only starts tile j after that head's
            // stage completed)
            float sp[32];
            if (nt0 * G > 16)
                race_bits32(so + nk + ta0 * G, nt0 * G, beta, sp);
            else
                race_bits16(so + nk + ta0 * G, nt0 * G, beta, sp);
            float dacc[4] = {0.0f, 0.0f, 0.0f, 0.0f};  // independent chains
            chunk_den<G, T>(sp, nt0, Asm + ta0 * R, dacc);
            // the second chunk's factors wait for the P V product: kept as
            // fp16 pairs (factors lie in (0.11, 0.89); relative rounding
            // 2^-11, below the bf16 rounding of the features they make)
            uint32_t sp1[8];
            if constexpr (T * G <= 16) {
                if (nt1 > 0) {
                    race_bits16(so + nk + ta1 * G, nt1 * G, beta, sp + 16);
                    chunk_den<G, T>(sp + 16, nt1, Asm + ta1 * R, dacc);
#pragma unroll
                    for (int q = 0; q < 8; ++q)
                        sp1[q] = pack_f16x2(sp[16 + 2 * q], sp[17 + 2 * q]);
                }
            }
            const float den = (dacc[0] + dacc[1]) + (dacc[2] + dacc[3]);
            // softmax over this half's key columns
            const int klo = b < 128 ? (row / b) * b : 0;
            const int khi = b < 128 ? klo + b : nk;
            float mxa[4] = {-INFINITY, -INFINITY, -INFINITY, -INFINITY};
            const bool masked = b < 128;
            // pass 0 of a tile whose window starts before the sequence
            const bool valid0 = !WIN || pass_valid(p0, 0);
            // SEL: this row's selected candidates among this half's 64 keys
            // of pass ps (bit k of the 64-bit word: key kbeg + k)
            const size_t selrow = (size_t)bh * N + (size_t)min(qpos, N - 1);
            const int selw = tk_c * b / 32;
            auto selbits = [&](int ps) -> unsigned long long {
                if (!SEL) return ~0ull;
                const uint32_t *w = selmask + selrow * selw + 4 * ps + 2 * half;
                return (unsigned long long)w[0] |
                       ((unsigned long long)w[1] << 32);
            };
            const unsigned long long sb0 = selbits(0);
#pragma unroll
            for (int c = 0; c < nk / 2; c += 16) {
                uint32_t v[16];
                tmem_ld16(so + kbeg + c, v);
                tmem_wait_ld();
#pragma unroll
                for (int jj = 0; jj < 16; ++jj) {
                    const int key = kbeg + c + jj;
                    if ((!WIN || valid0) &&
                        (!masked || (key >= klo && key < khi)) &&
                        (!SEL || ((sb0 >> (c + jj)) & 1ull)))
                        mxa[jj & 3] = fmaxf(mxa[jj & 3], __uint_as_float(v[jj]));
                }
            }
            float mx = fmaxf(fmaxf(mxa[0], mxa[1]), fmaxf(mxa[2], mxa[3]));
            xmax[g][half][row] = mx;
            xden[g][half][row] = den;
            named_sync(1 + g, 256);
            mx = fmaxf(xmax[g][0][row], xmax[g][1][row]);
            const float denf =
                (xden[g][0][row] + xden[g][1][row]) * (1.0f / (float)L);
            float M2 = mx * sl2e;
            float ls[4] = {0.0f, 0.0f, 0.0f, 0.0f};
#pragma unroll
            for (int c = 0; c < nk / 2; c += 32) {
                uint32_t pk16[16];
#pragma unroll
                for (int hh = 0; hh < 2; ++hh) {
                    uint32_t v[16];
                    tmem_ld16(so + kbeg + c + 16 * hh, v);
                    tmem_wait_ld();
#pragma unroll
                    for (int jj = 0; jj < 16; jj += 2) {
                        const int key = kbeg + c + 16 * hh + jj;
                        float a0 = ex2_approx(
                            fmaf(__uint_as_float(v[jj]), sl2e, -M2));
                        float a1 = ex2_approx(
                            fmaf(__uint_as_float(v[jj + 1]), sl2e, -M2));
                        if (masked) {
                            a0 = (key >= klo && key < khi) ? a0 : 0.0f;
                            a1 = (key + 1 >= klo && key + 1 < khi) ? a1 : 0.0f;
                        }
                        if (WIN && !valid0) a0 = a1 = 0.0f;
                        if (SEL) {
                            const int kl = c + 16 * hh + jj;  // in the half
                            a0 = ((sb0 >> kl) & 1ull) ? a0 : 0.0f;
                            a1 = ((sb0 >> (kl + 1)) & 1ull) ? a1 : 0.0f;
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
            bool pass_fail = false;
#pragma unroll
            for (int ps = 1; ps < NPASS; ++ps) {
                // the previous pass's P goes to its P V product; this pass
                // scores the next 128 keys into the same columns
                tmem_wait_st();
                tc_fence_before();
                mbar_arrive(&bars.p_full[g]);
                if (!wwait(&bars.s_full[g], (k * NPASS + ps) & 1, 56)) {
                    pass_fail = true;
                    break;
                }
                tc_fence_after();
                // the K buffer is free again: the next pass's keys, or after
                // the last pass the next tile's queries and keys
                if (ps + 1 < NPASS) {
                    if (!issue_k(j, ps + 1)) {
                        pass_fail = true;
                        break;
                    }
                } else if (j + 1 < ntiles && !issue_qk(j + 1)) {
                    pass_fail = true;
                    break;
                }
                const bool pvalid = !WIN || pass_valid(p0, ps);
                const unsigned long long sbp = selbits(ps);
                float mxb[4] = {-INFINITY, -INFINITY, -INFINITY, -INFINITY};
                if (!WIN || pvalid) {
#pragma unroll
                    for (int c = 0; c < nk / 2; c += 16) {
                        uint32_t v[16];
                        tmem_ld16(so + kbeg + c, v);
                        tmem_wait_ld();
#pragma unroll
                        for (int jj = 0; jj < 16; ++jj)
                            if (!SEL || ((sbp >> (c + jj)) & 1ull))
                                mxb[jj & 3] = fmaxf(mxb[jj & 3],
                                                    __uint_as_float(v[jj]));
                    }
                }
                xmax[g][half][row] =
                    fmaxf(fmaxf(mxb[0], mxb[1]), fmaxf(mxb[2], mxb[3]));
                named_sync(1 + g, 256);
                const float M2b =
                    fmaxf(xmax[g][0][row], xmax[g][1][row]) * sl2e;
                // online softmax: keep the running reference unless the
                // row's max grew by more than 2^8; then rescale the
                // accumulator (the previous P V product is complete: these
                // scores waited for it) and the running sum. From an empty
                // start (M2 = -inf) the factor is 0.
                const bool need = M2b > M2 + 8.0f;
                const float f = need ? ex2_approx(M2 - M2b) : 1.0f;
                if (__any_sync(0xffffffffu, need)) {
#pragma unroll
                    for (int c = 0; c < 64; c += 16) {
                        if (c < (d >> 1)) {
                            uint32_t v[16];
                            tmem_ld16(so + nk + half * (d >> 1) + c, v);
                            tmem_wait_ld();
#pragma unroll
                            for (int q = 0; q < 16; ++q)
                                v[q] = __float_as_uint(__uint_as_float(v[q]) * f);
                            tmem_st16(so + nk + half * (d >> 1) + c, v);
                        }
                    }
                }
                if (need) {
                    lsum *= f;
                    M2 = M2b;
                }
                float lb[4] = {0.0f, 0.0f, 0.0f, 0.0f};
#pragma unroll
                for (int c = 0; c < nk / 2; c += 32) {
                    uint32_t pk16[16];
#pragma unroll
                    for (int hh = 0; hh < 2; ++hh) {
                        uint32_t v[16];
                        tmem_ld16(so + kbeg + c + 16 * hh, v);
                        tmem_wait_ld();
#pragma unroll
                        for (int jj = 0; jj < 16; jj += 2) {
                            float a0 = ex2_approx(
                                fmaf(__uint_as_float(v[jj]), sl2e, -M2));
                            float a1 = ex2_approx(
                                fmaf(__uint_as_float(v[jj + 1]), sl2e, -M2));
                            if (WIN && !pvalid) a0 = a1 = 0.0f;
                            if (SEL) {
                                const int kl = c + 16 * hh + jj;
                                a0 = ((sbp >> kl) & 1ull) ? a0 : 0.0f;
                                a1 = ((sbp >> (kl + 1)) & 1ull) ? a1 : 0.0f;
                            }
                            lb[(jj >> 1) & 3] += a0 + a1;
                            pk16[8 * hh + (jj >> 1)] = pack_bf16x2(a0, a1);
                        }
                    }
                    tmem_st16(so + kbeg + (c >> 1), pk16);
                }
                xsum[g][half][row] = (lb[0] + lb[1]) + (lb[2] + lb[3]);
                tc_fence_before();
                named_sync(1 + g, 256);
                tc_fence_after();
                lsum += xsum[g][0][row] + xsum[g][1][row];
            }
            if (pass_fail) break;
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
            if (nt0 > 0) write_phi_chunk<G, T>(sp, nt0, ratio, so + cb0);
            tmem_wait_st();
            tc_fence_before();
            mbar_arrive(&bars.p_full[g]);
            if (r > nk) {
                if (!wwait(&bars.pv_done[g], k & 1, 52)) break;
                tc_fence_after();
                if constexpr (T * G <= 16) {
                    if (nt1 > 0) {
                        float f1[16];
#pragma unroll
                        for (int q = 0; q < 8; ++q)
                            unpack_f16x2(sp1[q], f1[2 * q], f1[2 * q + 1]);
                        write_phi_chunk<G, T>(f1, nt1, ratio, so + cb1);
                    }
                }
                tmem_wait_st();
                tc_fence_before();
                mbar_arrive(&bars.p2_full[g]);
            }
            if (!wwait(&bars.o_full[g], k & 1, 53)) break;
            tc_fence_after();
            // O = c1 acc as bf16, this half's d / 2 columns, staged in this
            // slot's V buffer (the P V product of the tile is complete) in
            // the swizzled panel layout, then copied out by the slot's 256
            // threads in whole rows (coalesced 16-byte stores). With an
            // fp32 output (o32) each thread stores its half row directly.
            const uint32_t sVg = sV0 + g * tileB;
            constexpr int kMaxHalf = 64;  // d / 2 for d = 128
#pragma unroll
            for (int c = 0; c < kMaxHalf; c += 16) {
                if (c < (d >> 1)) {
                    uint32_t v[16], ob[8];
                    tmem_ld16(so + nk + half * (d >> 1) + c, v);
                    tmem_wait_ld();
                    if constexpr (O32) {
                        if (qvalid) {
                            float4 *dst = reinterpret_cast<float4 *>(
                                o32 + tok * (size_t)d + half * (d >> 1) + c);
#pragma unroll
                            for (int q = 0; q < 4; ++q)
                                dst[q] = make_float4(
                                    c1e * __uint_as_float(v[4 * q]),
                                    c1e * __uint_as_float(v[4 * q + 1]),
                                    c1e * __uint_as_float(v[4 * q + 2]),
                                    c1e * __uint_as_float(v[4 * q + 3]));
                        }
                        continue;
                    }
#pragma unroll
                    for (int q = 0; q < 8; ++q)
                        ob[q] = pack_bf16x2(c1e * __uint_as_float(v[2 * q]),
                                            c1e * __uint_as_float(v[2 * q + 1]));
                    const int cidx = (half * (d >> 1) + c) >> 3;  // 16-B chunk
                    st_shared_v4(sVg + panel_offset(row, cidx, nk), ob[0],
                                 ob[1], ob[2], ob[3]);
                    st_shared_v4(sVg + panel_offset(row, cidx + 1, nk), ob[4],
                                 ob[5], ob[6], ob[7]);
                }
            }
            tc_fence_before();
            mbar_arrive(&bars.tmem_empty[g]);
            if (half == 0) {
                orow[g][row] = qvalid ? (int)tok : -1;
                if (qvalid) {
                    if (log_ds_out) log_ds_out[tok] = log_ds;
                    if (dlr_out) dlr_out[tok] = denf;
                    if (m_out) m_out[tok] = msp;
                }
            }
            named_sync(1 + g, 256);
            if constexpr (!O32) {
                const int ct = (cw & 7) * 32 + lane_id;  // 0..255
                const int cpr = d >> 3, rpp = 256 / cpr;
                const int crow = ct / cpr, cc = ct - crow * cpr;
                for (int rr = crow; rr < nk; rr += rpp) {
                    const int orr = orow[g][rr];
                    if (orr >= 0) {
                        const uint4 val =
                            ld_shared_v4(sVg + panel_offset(rr, cc, nk));
                        *reinterpret_cast<uint4 *>(ox + (size_t)orr * d +
                                                   cc * 8) = val;
                    }
                }
            }
            named_sync(1 + g, 256);  // the staging buffer is read
            if (cw == 8 * g && lane_id == 0) mbar_arrive(&bars.v_empty[g]);
        }
        cp_async_wait<0>();
    }
    tc_fence_before();
    __syncthreads();
    if (warp == kWsMmaWarp) tmem_dealloc(tm, 512);
}

}  // namespace

// 128-key passes per query tile, or 0 when no instantiation covers it:
// b <= 128 without neighbours: 1; b = 256: 2; neighbouring blocks (b of
// 128 or 256, gamma = 4): the (2 nb + 1) b / 128 passes of the window, 3 or
// 6 for nb = 1.
static int ws_passes(const Plan &P) {
    if (P.sel) {  // the candidate blocks, 128 keys per pass (b >= 128)
        if (P.gamma != 4 || (P.b != 128 && P.b != 256)) return 0;
        const int n = P.tk_c * P.b / 128;
        return n <= 4 ? n : 0;
    }
    if (P.nb == 0) return P.b <= 128 ? 1 : (P.b == 256 ? 2 : 0);
    if (P.nb != 1 || P.gamma != 4 || (P.b != 128 && P.b != 256)) return 0;
    return 3 * (P.b / 128);
}

bool ws_supported(const Plan &P) {
    // a half's chunks: the first may use up to 32 projection columns, the
    // second (buckets past 128) at most 16, i.e. gamma >= 4 when r > 128;
    // row numbers in int
    const long rows = (long)P.N * P.BH;  // row numbers are int
    // fp32 output is instantiated for gamma = 4; other gamma with out_fp32
    // run the CUDA-core block kernel
    if (P.o32 && P.gamma != 4) return false;
    return tc_supported(P) && ws_passes(P) > 0 &&
           (P.gamma >= 4 || P.r <= 128) && rows < (1L << 31);
}

cudaError_t launch_block_attn_ws(
    const Plan &P, const void *q, const void *k, const void *v,
    const uint16_t *w_bf16, const int32_t *perm_q, const int32_t *perm_k,
    const float *A, const uint16_t *Bh, const float *lambda_tok,
    const float *gates, void *o, float *log_d_sparse, float *d_lr,
    float *m_sparse, DeviceStatus *status, cudaStream_t st,
    const int32_t *cand, const uint32_t *selmask) {
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
    CUtensorMap tmW, tmB;
    cudaError_t e = make_tma_map_bf16(&tmW, w_bf16, (uint64_t)P.H * P.Lg_pad,
                                      P.d, (uint32_t)P.Lg_pad);
    if (e == cudaSuccess)
        e = make_tma_map_bf16(&tmB, Bh, (uint64_t)P.BH * P.r, P.d,
                              (uint32_t)P.r);
    if (e != cudaSuccess) return e;
    auto launch = [&](auto kern) {
        cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             (int)smem);
        kern<<<grid, kWsThreads, smem, st>>>(
            (const uint16_t *)q, (const uint16_t *)k, (const uint16_t *)v,
            tmW, tmB, perm_q, perm_k, A, lambda_tok, gates,
            P.o32 ? nullptr : (uint16_t *)o, P.o32 ? (float *)o : nullptr,
            log_d_sparse, d_lr, m_sparse, P.N, P.d, P.H, P.b, P.nb, P.L, lg,
            P.beta, P.eps, P.scale, P.lambda, P.fusion_mode, tiles_per_head,
            total, status, cand, selmask, P.tk_c);
        return cudaGetLastError();
    };
    const int passes = ws_passes(P);
    if (P.o32) {  // fp32 output: gamma = 4 (ws_supported)
        if (P.sel) {
            switch (passes) {
                case 1: return launch(k_block_attn_ws<4, 1, 2, true>);
                case 2: return launch(k_block_attn_ws<4, 2, 2, true>);
                case 3: return launch(k_block_attn_ws<4, 3, 2, true>);
                case 4: return launch(k_block_attn_ws<4, 4, 2, true>);
                default: return cudaErrorInvalidValue;
            }
        }
        if (passes == 3) return launch(k_block_attn_ws<4, 3, 1, true>);
        if (passes == 6) return launch(k_block_attn_ws<4, 6, 1, true>);
        if (P.gamma != 4) return cudaErrorInvalidValue;
        return P.b > 128 ? launch(k_block_attn_ws<4, 2, 0, true>)
                         : launch(k_block_attn_ws<4, 1, 0, true>);
    }
    if (P.sel) {
        switch (passes) {
            case 1: return launch(k_block_attn_ws<4, 1, 2>);
            case 2: return launch(k_block_attn_ws<4, 2, 2>);
            case 3: return launch(k_block_attn_ws<4, 3, 2>);
            case 4: return launch(k_block_attn_ws<4, 4, 2>);
            default: return cudaErrorInvalidValue;
        }
    }
    if (passes == 3) return launch(k_block_attn_ws<4, 3, 1>);
    if (passes == 6) return launch(k_block_attn_ws<4, 6, 1>);
    switch (P.gamma) {
        case 1: return P.b > 128 ? launch(k_block_attn_ws<1, 2, 0>) : launch(k_block_attn_ws<1, 1, 0>);
        case 2: return P.b > 128 ? launch(k_block_attn_ws<2, 2, 0>) : launch(k_block_attn_ws<2, 1, 0>);
        case 3: return P.b > 128 ? launch(k_block_attn_ws<3, 2, 0>) : launch(k_block_attn_ws<3, 1, 0>);
        case 4: return P.b > 128 ? launch(k_block_attn_ws<4, 2, 0>) : launch(k_block_attn_ws<4, 1, 0>);
        case 5: return P.b > 128 ? launch(k_block_attn_ws<5, 2, 0>) : launch(k_block_attn_ws<5, 1, 0>);
        case 6: return P.b > 128 ? launch(k_block_attn_ws<6, 2, 0>) : launch(k_block_attn_ws<6, 1, 0>);
        default: return cudaErrorInvalidValue;
    }
}

}  // namespace elsaa
