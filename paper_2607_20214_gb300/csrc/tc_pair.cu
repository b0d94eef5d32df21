// Block attention for key blocks of 256 (b = 256, d_h = 128, gamma = 4) on
// CTA pairs: the sortLSH block step (Algorithm "sortLSH Sparse Exact
// Attention Branch"), the RACE readout (Algorithm "RACE Low-Rank Attention
// Branch" steps 9-10) and the fusion of Eq. (5)-(6), the same arithmetic as
// the one-CTA kernel of tc_ws.cu.
//
// The two 128-query tiles of one sorted block attend the same 256 keys, so
// a cluster of two CTAs on neighbouring SMs takes one block at a time: the
// even CTA the block's first 128 queries, the odd CTA the other 128. Every
// product is one cta_group::2 MMA (M = 256: each CTA's 128 query rows in its
// own tensor memory) whose B operand is split by columns between the CTAs:
//   scores   S = Q [K; W]^T: each CTA gathers 64 of the pass's 128 keys and
//            holds 32 of the 64 RACE plane rows (its row half's tables);
//   P V:     each CTA gathers its 64 of the 128 value columns;
//   Phi' B:  each CTA holds its 64 columns of the bf16 B summary.
// So each SM gathers half a block's keys and values instead of all of them,
// and the freed shared memory double-buffers the query tile and holds one
// key and one value buffer per pass.
//
// Roles (640 threads per CTA): warps 0-15 compute (two TMEM slots of 256
// columns, slot g takes the CTA's blocks of local index = g mod 2; within a
// slot warps w and w + 4 split each row's keys, tables and output columns
// in halves), warp 16 issues every MMA in the even CTA and relays the odd
// CTA's readiness to it, warp 17 resolves row numbers, warp 18 loads the
// per-head planes and summaries with TMA, warp 19 gathers values.
//
// TMEM columns of a slot (same layout in both CTAs): pass 0 scores keys
// [0, 64) at [0, 64), the projections of row half 0's tables at [64, 96),
// keys [64, 128) at [96, 160), row half 1's projections at [160, 192);
// pass 1 scores keys [0, 64) at [0, 64), keys [64, 128) at [64, 128); P of
// row half h in quarter 2h ([64h, 64h + 32)); the output accumulator at
// [128, 256); the pre-scaled features as in the one-CTA kernel.
//
// Every hand-off is an mbarrier with a bounded wait; the odd CTA's
// arrivals reach the even CTA's barriers through the relay (one remote
// arrival per phase), the MMA completions reach both CTAs by multicast.
#include "device_common.cuh"
#include "tc_common.cuh"
#include "tc_race.cuh"

namespace elsaa {

namespace {

using namespace tc;

constexpr int kPrThreads = 640;
constexpr int kPrMmaWarp = 16;
constexpr int kPrLoaders = 32;
constexpr int kPrNK = 128;   // keys per pass, query rows per CTA
constexpr int kPrNP = 2;     // passes per block (b = 256)
constexpr int kPrD = 128;    // head dimension
constexpr int kPrKRows0 = 96;  // pass-0 key buffer: 64 keys + 32 plane rows
constexpr int kPrKRows1 = 64;  // pass-1 key buffer: 64 keys

struct PrBars {
    // copies, relayed: the even CTA's copy also counts the odd CTA's phase
    uint64_t q_full[2], k_full[kPrNP], v_full[kPrNP], wb_full;
    // compute hand-offs: the odd CTA's slot arrives once on the even CTA's
    // barrier after its own named barrier
    uint64_t tmem_empty[2], p_full[2], p2_full[2];
    // MMA completions, committed to both CTAs
    uint64_t s_full[2], pv0_done[2], pv_done[2], o_full[2], v_empty[kPrNP];
    uint64_t head_done;
    // local
    uint64_t idx_full[2], idx_empty[2];
};
constexpr int kPrRelayed = 2 + kPrNP + kPrNP + 1;  // copy barriers

template <bool O32>
__global__ void __launch_bounds__(kPrThreads, 1)
    k_block_attn_pair(const uint16_t *__restrict__ qx,
                      const uint16_t *__restrict__ kx,
                      const uint16_t *__restrict__ vx,
                      const __grid_constant__ CUtensorMap tmW,
                      const __grid_constant__ CUtensorMap tmB,
                      const int32_t *__restrict__ perm_q,
                      const int32_t *__restrict__ perm_k,
                      const float *__restrict__ Ag,
                      const float *__restrict__ lambda_tok,
                      const float *__restrict__ gates,
                      uint16_t *__restrict__ ox, float *__restrict__ o32,
                      float *__restrict__ log_ds_out,
                      float *__restrict__ dlr_out, float *__restrict__ m_out,
                      int N, int H, int L, int Lg_pad, float beta, float eps,
                      float scale, float lambda, int mode, int blocks_per_head,
                      long total_blocks, DeviceStatus *status) {
    constexpr int G = 4, R = 16, nk = kPrNK, d = kPrD, NP = kPrNP;
    extern __shared__ unsigned char smem_raw[];
    __shared__ PrBars bars;
    __shared__ uint32_t tbase;
    __shared__ int abort_flag;
    __shared__ float xmax[2][2][128], xsum[2][2][128], xden[2][2][128];
    // row numbers of a block's queries (this CTA's 128) and of this CTA's
    // 64 keys of each pass, per block parity
    __shared__ __align__(16) int qrow[2][128];
    __shared__ __align__(16) int krow[2][NP][64];
    __shared__ __align__(16) int vrow[128];  // value loader: the pass's keys
    volatile int *abort = &abort_flag;
    const int tid = threadIdx.x, warp = tid >> 5, lane_id = tid & 31;
    const uint32_t crank = cluster_rank();  // 0: issues the MMAs
    const bool leader = crank == 0;
    const int r = L * R;
    const long pair = blockIdx.x >> 1, npairs = gridDim.x >> 1;
    const long b_begin = total_blocks * pair / npairs;
    const long b_end = total_blocks * (pair + 1) / npairs;
    const int nblk = (int)(b_end - b_begin);
    const int bb = (int)b_begin;  // block indices fit in int (host check)
    auto blk_head = [=](int j) { return (bb + j) / blocks_per_head; };
    // sorted position of this CTA's first query of block j
    auto blk_pos = [=](int j) {
        return (bb + j) % blocks_per_head * 256;
    };
    auto new_head = [=](int j) {
        return j == 0 || (bb + j) % blocks_per_head == 0;
    };
    auto last_of_head = [=](int j) {
        return j == nblk - 1 || (bb + j + 1) % blocks_per_head == 0;
    };

    // shared memory: two query tiles, the pass-0 key buffer (64 keys and
    // this CTA's 32 plane rows), the pass-1 key buffer, one value buffer per
    // pass (128 keys x this CTA's 64 columns), this CTA's 64 columns of the
    // B summary, the A summary
    const uint32_t tileQ = (uint32_t)nk * d * 2u;
    const uint32_t base = align1k(smem_u32(smem_raw));
    const uint32_t sQ = base;
    const uint32_t sK0 = sQ + 2 * tileQ;
    const uint32_t sK1 = sK0 + kPrKRows0 * d * 2;
    const uint32_t sV = sK1 + kPrKRows1 * d * 2;
    const uint32_t sB = sV + NP * 16384u;
    const uint32_t sA = sB + align1k((uint32_t)r * 128u);
    const float *Asm = reinterpret_cast<const float *>(
        smem_raw + (sA - smem_u32(smem_raw)));
    auto kbuf = [=](int p) { return p == 0 ? sK0 : sK1; };
    auto krows = [=](int p) { return p == 0 ? kPrKRows0 : kPrKRows1; };

    if (warp == kPrMmaWarp) tmem_alloc_pair(&tbase, 512);
    if (tid == 0) {
        const uint32_t x = leader ? 1u : 0u;  // the relayed odd-CTA phase
        for (int s = 0; s < 2; ++s) {
            mbar_init(&bars.q_full[s], 256 + x);
            mbar_init(&bars.tmem_empty[s], 256 + x);
            mbar_init(&bars.p_full[s], 256 + x);
            mbar_init(&bars.p2_full[s], 256 + x);
            mbar_init(&bars.s_full[s], 1);
            mbar_init(&bars.pv0_done[s], 1);
            mbar_init(&bars.pv_done[s], 1);
            mbar_init(&bars.o_full[s], 1);
            mbar_init(&bars.idx_full[s], kPrLoaders);
            mbar_init(&bars.idx_empty[s], 256 * (1 + NP));
        }
        for (int p = 0; p < NP; ++p) {
            mbar_init(&bars.k_full[p], 256 + x);
            mbar_init(&bars.v_full[p], kPrLoaders + x);
            mbar_init(&bars.v_empty[p], 1);
        }
        mbar_init(&bars.wb_full, 1 + x);
        mbar_init(&bars.head_done, 1);
        abort_flag = 0;
        fence_mbar_init();
    }
    tc_fence_before();
    __syncthreads();
    cluster_sync();  // both CTAs' barriers exist before any remote arrival
    tc_fence_after();
    const uint32_t tm = tbase;

    // global row numbers of the 4 sorted positions pos.. pos + 3 of one
    // head (rowbase = its first row); an entry outside [0, N) is read as
    // row 0 (the orders come from the sort); the checked build records it
    auto rows4 = [=](const int32_t *pm, int pos, int rowbase) {
        int4 v;  // pos + 3 < N: N is a multiple of 256
        if (((uintptr_t)(pm + pos) & 15u) == 0) {
            v = *reinterpret_cast<const int4 *>(pm + pos);
        } else {
            v = make_int4(pm[pos], pm[pos + 1], pm[pos + 2], pm[pos + 3]);
        }
        auto fix = [=](int u) {
            if (u < 0 || u >= N) {
#ifdef ELSAA_CHECKED
                report(status, kDevPermRange, 14, rowbase / N, u);
#endif
                u = 0;
            }
            return rowbase + u;
        };
        return make_int4(fix(v.x), fix(v.y), fix(v.z), fix(v.w));
    };

    if (warp > kPrMmaWarp) {
        // ------------------------------------------------------------ loaders
        const int role = warp - kPrMmaWarp - 1;
        const int lt = lane_id;
        auto lwait = [=](uint64_t *bar, uint32_t par, int site) {
            return __all_sync(0xffffffffu,
                              mbar_wait_or_abort(bar, par, abort, status,
                                                 site));
        };
        if (role == 0) {
            // row numbers of block j (this CTA's queries, its keys of each
            // pass) into slot j & 1 once block j - 2's gathers went out
            for (int j = 0; j < nblk; ++j) {
                const int t = j & 1, bh = blk_head(j), pos = blk_pos(j);
                if (j >= 2 &&
                    !lwait(&bars.idx_empty[t], ((j >> 1) - 1) & 1, 70))
                    break;
                *reinterpret_cast<int4 *>(&qrow[t][4 * lt]) =
                    rows4(perm_q + (size_t)bh * N, pos + 128 * crank + 4 * lt,
                          bh * N);
                if (lt < 16) {
#pragma unroll
                    for (int p = 0; p < NP; ++p)
                        *reinterpret_cast<int4 *>(&krow[t][p][4 * lt]) =
                            rows4(perm_k + (size_t)bh * N,
                                  pos + 128 * p + 64 * crank + 4 * lt,
                                  bh * N);
                }
                __syncwarp();
                mbar_arrive(&bars.idx_full[t]);
            }
        } else if (role == 1) {
            // per head, TMA: this CTA's 32 plane rows (its row half's tables:
            // rows [16 c, 16 c + 16) and [32 + 16 c, 48 + 16 c) of the head's
            // planes) under the pass-0 keys, its 64 columns of the B summary,
            // the A summary
            int hc = 0;
            for (int j = 0; j < nblk; ++j) {
                if (!new_head(j)) continue;
                const int bh = blk_head(j);
                if (j > 0 && !lwait(&bars.head_done, (hc - 1) & 1, 71)) break;
                if (lt == 0) {
                    mbar_expect_tx(&bars.wb_full,
                                   32u * d * 2u + (uint32_t)r * 128u +
                                       (uint32_t)r * 4u);
                    const int w0 = (bh % H) * Lg_pad + 16 * (int)crank;
                    for (int pn = 0; pn < d / 64; ++pn) {
                        const uint32_t dst = sK0 + pn * kPrKRows0 * 128;
                        tma_load_2d(dst + 64 * 128, &tmW, 64 * pn, w0,
                                    &bars.wb_full);
                        tma_load_2d(dst + 80 * 128, &tmW, 64 * pn, w0 + 32,
                                    &bars.wb_full);
                    }
                    tma_load_2d(sB, &tmB, 64 * (int)crank, bh * r,
                                &bars.wb_full);
                    bulk_load(sA, Ag + (size_t)bh * r, (uint32_t)r * 4u,
                              &bars.wb_full);
                }
                __syncwarp();
                ++hc;
            }
        } else {
            // values: for each pass, the pass's 128 keys, this CTA's 64
            // columns (128 bytes of each row) into the pass's buffer once
            // the previous block's P V product of that pass is done
            const int lrow = lt >> 3, lc = lt & 7;  // 4 rows per instruction
            bool go = true;
            for (int j = 0; j < nblk && go; ++j) {
                const int bh = blk_head(j), pos = blk_pos(j);
                for (int p = 0; p < NP; ++p) {
                    __syncwarp();  // the previous rows are all read
                    *reinterpret_cast<int4 *>(&vrow[4 * lt]) =
                        rows4(perm_k + (size_t)bh * N, pos + 128 * p + 4 * lt,
                              bh * N);
                    __syncwarp();
                    if (j >= 1 &&
                        !lwait(&bars.v_empty[p], (j - 1) & 1, 72)) {
                        go = false;
                        break;
                    }
                    const uint32_t dst = sV + p * 16384u;
                    for (int row = lrow; row < nk; row += 4)
                        cp_async16(dst + panel_offset(row, lc, nk),
                                   vx + (size_t)vrow[row] * d +
                                       64 * (int)crank + lc * 8);
                    cp_async_mbar_arrive(&bars.v_full[p]);
                }
            }
            cp_async_wait<0>();
        }
    } else if (warp == kPrMmaWarp) {
        if (!leader) {
            // ------------------------------------------------------ relay
            // Each phase of this CTA's copy barriers (cp.async and TMA
            // completions, which can only arrive locally) completes here
            // first, then counts once more on the even CTA's copy. A phase
            // cannot complete twice before it is relayed: the next one needs
            // MMAs that wait for this relay.
            if (lane_id == 0) {
                uint64_t *bar[kPrRelayed] = {
                    &bars.q_full[0], &bars.q_full[1], &bars.k_full[0],
                    &bars.k_full[1], &bars.v_full[0], &bars.v_full[1],
                    &bars.wb_full};
                const int in0 = (nblk + 1) / 2, in1 = nblk / 2;  // per slot
                int heads = 0;
                for (int j = 0; j < nblk; ++j) heads += new_head(j) ? 1 : 0;
                const int want[kPrRelayed] = {in0,  in1,  nblk, nblk,
                                              nblk, nblk, heads};
                int done[kPrRelayed];
                int left = 0;
                for (int i = 0; i < kPrRelayed; ++i) {
                    done[i] = 0;
                    left += want[i];
                }
                unsigned long long t_last = global_ns();
                while (left > 0) {
                    bool did = false;
                    for (int i = 0; i < kPrRelayed; ++i) {
                        if (done[i] < want[i] &&
                            mbar_test(bar[i], (uint32_t)done[i] & 1u)) {
                            // this CTA's cp.async data -> the pair's MMAs
                            fence_proxy_async_smem();
                            mbar_arrive_remote(bar[i], 0);
                            ++done[i];
                            --left;
                            did = true;
                        }
                    }
                    if (did) {
                        t_last = global_ns();
                    } else {
                        if (*abort) break;
                        if (global_ns() - t_last > kWaitLimitNs) {
                            *abort = 1;
                            record_timeout(status, 73);
                            break;
                        }
                    }
                }
            }
        } else if (lane_id == 0 && nblk > 0) {
            // ------------------------------------------------- MMA issue
            // Event driven as in the one-CTA kernel, over units (block,
            // pass): the oldest block's second feature part first, then
            // P V (with the first feature part after the last pass), then
            // the next scores. Pass 1's scores reuse the S columns and wait
            // for pass 0's P V product.
            const uint32_t id_sp = idesc_bf16(256, nk + 64, false, false);
            const uint32_t id_s = idesc_bf16(256, nk, false, false);
            const uint32_t id_o = idesc_bf16(256, d, false, true);
            const int r0 = min(r, nk);
            const bool two_parts = r > nk;
            const int nunits = nblk * NP;
            int us = 0, up = 0, i2 = 0, blocks_pv = 0, hc = 0;
            unsigned long long t_last = global_ns();
            while ((two_parts ? i2 : blocks_pv) < nblk) {
                bool did = false;
                if (two_parts && i2 < blocks_pv) {
                    const int s = i2 & 1;
                    const uint32_t so = tm + 256u * s;
                    if (mbar_test(&bars.p2_full[s], (i2 >> 1) & 1)) {
                        tc_fence_after();
                        for (int kk = 0; kk < (r - nk) / 16; ++kk)
                            mma_pair_ts(so + nk, so + quarter_col(kk, 0),
                                        smem_desc(sB + (uint32_t)nk * 128 +
                                                      kk * 2048,
                                                  (uint32_t)r * 128, 1024),
                                        id_o, 1);
                        mma_commit_pair(&bars.o_full[s]);
                        if (last_of_head(i2)) mma_commit_pair(&bars.head_done);
                        ++i2;
                        did = true;
                    }
                }
                if (up < us) {
                    const int j = up / NP, p = up - j * NP, s = j & 1;
                    const int su = (j >> 1) * NP + p;  // unit within slot
                    const uint32_t so = tm + 256u * s;
                    if (mbar_test(&bars.p_full[s], su & 1) &&
                        mbar_test(&bars.v_full[p], j & 1)) {
                        fence_proxy_async_smem();  // cp.async data -> MMA
                        tc_fence_after();
                        const uint32_t vb = sV + p * 16384u;
                        for (int kk = 0; kk < nk / 16; ++kk)  // O (+)= P V
                            mma_pair_ts(so + nk, so + quarter_col(kk, 0),
                                        smem_desc(vb + kk * 2048,
                                                  (uint32_t)nk * 128, 1024),
                                        id_o, p > 0 || kk > 0);
                        mma_commit_pair(&bars.v_empty[p]);
                        if (p < NP - 1) {
                            mma_commit_pair(&bars.pv0_done[s]);
                        } else {
                            for (int kk = 0; kk < r0 / 16; ++kk)  // + Phi' B
                                mma_pair_ts(so + nk, so + quarter_col(kk, 32),
                                            smem_desc(sB + kk * 2048,
                                                      (uint32_t)r * 128,
                                                      1024),
                                            id_o, 1);
                            if (two_parts) {
                                mma_commit_pair(&bars.pv_done[s]);
                            } else {
                                mma_commit_pair(&bars.o_full[s]);
                                if (last_of_head(j))
                                    mma_commit_pair(&bars.head_done);
                            }
                            ++blocks_pv;
                        }
                        ++up;
                        did = true;
                    }
                }
                // a new head's planes and summaries replace the old ones
                // only after head_done: its first scores wait until every
                // MMA of the previous head is issued
                const int js = us / NP, ps = us - js * NP;
                const bool nh = ps == 0 && new_head(js);
                if (us < nunits &&
                    !(nh && js > 0 && (two_parts ? i2 : blocks_pv) < js)) {
                    const int s = js & 1;
                    const uint32_t so = tm + 256u * s;
                    bool ready = mbar_test(&bars.k_full[ps], js & 1);
                    if (ready && ps == 0)
                        ready = mbar_test(&bars.q_full[s],
                                                  (js >> 1) & 1) &&
                                (js < 2 ||
                                 mbar_test(&bars.tmem_empty[s],
                                                   ((js >> 1) - 1) & 1)) &&
                                (!nh || mbar_test(&bars.wb_full,
                                                          hc & 1));
                    if (ready && ps > 0)  // S columns hold P of pass ps - 1
                        ready = mbar_test(&bars.pv0_done[s],
                                          ((js >> 1) * (NP - 1) + ps - 1) &
                                              1);
                    if (ready) {
                        if (nh) ++hc;
                        fence_proxy_async_smem();  // cp.async data -> MMA
                        tc_fence_after();
                        const uint32_t kb = kbuf(ps);
                        const int kr = krows(ps);
                        for (int kk = 0; kk < d / 16; ++kk) {
                            const uint32_t oq =
                                (kk >> 2) * 128 * 128 + (kk & 3) * 32;
                            const uint32_t okw =
                                (kk >> 2) * kr * 128 + (kk & 3) * 32;
                            // pass 0: scores and projections (N = 192);
                            // pass 1: scores only
                            mma_pair_ss(so,
                                        smem_desc(sQ + s * tileQ + oq, 16,
                                                  1024),
                                        smem_desc(kb + okw, 16, 1024),
                                        ps == 0 ? id_sp : id_s, kk > 0);
                        }
                        mma_commit_pair(&bars.s_full[s]);
                        ++us;
                        did = true;
                    }
                }
                if (did) {
                    t_last = global_ns();
                } else {
                    if (*abort) break;
                    if (global_ns() - t_last > kWaitLimitNs) {
                        *abort = 1;
                        record_timeout(status, 74);
                        break;
                    }
                }
            }
        }
        __syncwarp();
    } else {
        // ------------------------------------------------------ compute groups
        // warps 0-7: slot 0, warps 8-15: slot 1; within a slot, warps
        // (w, w + 4) share TMEM lanes and split each row in two halves: half
        // h takes keys [64 h, 64 h + 64) of each pass (the keys this CTA's
        // half of the pair gathered when h equals its rank), the tables of
        // the 64-bucket chunks h and h + 2 and output columns [64 h, 64 h +
        // 64).
        const int cw = warp;
        const int g = cw >> 3;
        const int half = (cw >> 2) & 1;
        const int row = (warp & 3) * 32 + lane_id;  // query row = TMEM lane
        const uint32_t lane = (uint32_t)((warp & 3) * 32) << 16;
        constexpr int T = 64 / R;  // tables per 64-bucket chunk
        const int ta0 = min(half * T, L), nt0 = min(ta0 + T, L) - ta0;
        const int ta1 = min((half + 2) * T, L), nt1 = min(ta1 + T, L) - ta1;
        const uint32_t cb0 = half ? 96u : 32u, cb1 = half ? 64u : 0u;
        const float sl2e = scale * kLog2e;
        auto wwait = [=](uint64_t *bar, uint32_t par, int site) {
            const bool ok = mbar_wait_or_abort(bar, par, abort, status, site);
            return named_sync_and(1 + g, 256, ok);
        };
        const int ct = (cw & 7) * 32 + lane_id;  // 0..255 within the slot
        // a hand-off to the MMA issuer: every thread of the even CTA's slot
        // arrives; the odd CTA's slot meets at its named barrier and one
        // thread arrives on the even CTA's barrier
        auto signal = [&](uint64_t *bar) {
            if (leader) {
                mbar_arrive(bar);
            } else {
                named_sync(1 + g, 256);
                if (ct == 0) mbar_arrive_remote(bar, 0);
            }
        };
        const int crow = ct >> 4, cc = ct & 15;  // 16 chunks per row
        // block j's queries into query buffer j & 1 (8 copies a thread)
        auto gather_q = [&](int j) -> bool {
            if (!wwait(&bars.idx_full[j & 1], (j >> 1) & 1, 75)) return false;
            const int *rows = qrow[j & 1];
            const uint32_t dst = sQ + (j & 1) * tileQ;
            for (int rr = crow; rr < nk; rr += 16)
                cp_async16(dst + panel_offset(rr, cc, nk),
                           qx + (size_t)rows[rr] * d + cc * 8);
            cp_async_mbar_arrive(&bars.q_full[j & 1]);
            mbar_arrive(&bars.idx_empty[j & 1]);
            return true;
        };
        // this CTA's 64 keys of block j's pass p into key buffer p
        auto gather_k = [&](int j, int p) -> bool {
            if (!wwait(&bars.idx_full[j & 1], (j >> 1) & 1, 76)) return false;
            const int *rows = krow[j & 1][p];
            const uint32_t dst = kbuf(p);
            const int ld = krows(p);
            for (int rr = crow; rr < 64; rr += 16)
                cp_async16(dst + panel_offset(rr, cc, ld),
                           kx + (size_t)rows[rr] * d + cc * 8);
            cp_async_mbar_arrive(&bars.k_full[p]);
            mbar_arrive(&bars.idx_empty[j & 1]);
            return true;
        };
        bool started = true;
        if (nblk > 0) {
            if (g == 0)
                started = gather_q(0) && gather_k(0, 0) && gather_k(0, 1);
            else if (nblk > 1)
                started = gather_q(1);
        }
        for (int j = g; started && j < nblk; j += 2) {
            const int k = j >> 1;
            const uint32_t so = tm + 256u * g + lane;
            const int bh = blk_head(j);
            const int qpos = blk_pos(j) + 128 * (int)crank + row;
            int qi = perm_q[(size_t)bh * N + qpos];  // prefetch
            if (!wwait(&bars.s_full[g], (k * NP) & 1, 77)) break;
            tc_fence_after();
            // this half's raw projections (pass 0 writes them where pass 0's
            // P and the output accumulator go): the per-bit factors and Den
            // are computed once pass 0's P is handed to its P V product
            uint32_t pr[32];
            const uint32_t pcol = 64u + 96u * half;  // this half's projections
            tmem_ld16(so + pcol, *reinterpret_cast<uint32_t(*)[16]>(pr));
            tmem_ld16(so + pcol + 16,
                      *reinterpret_cast<uint32_t(*)[16]>(pr + 16));
            tmem_wait_ld();
            // pass 0: this half's 64 key columns start at 96 h
            const uint32_t kc0 = 96u * half;
            float mxa[4] = {-INFINITY, -INFINITY, -INFINITY, -INFINITY};
#pragma unroll
            for (int c = 0; c < 64; c += 16) {
                uint32_t v[16];
                tmem_ld16(so + kc0 + c, v);
                tmem_wait_ld();
#pragma unroll
                for (int jj = 0; jj < 16; ++jj)
                    mxa[jj & 3] = fmaxf(mxa[jj & 3], __uint_as_float(v[jj]));
            }
            float mx = fmaxf(fmaxf(mxa[0], mxa[1]), fmaxf(mxa[2], mxa[3]));
            xmax[g][half][row] = mx;
            named_sync(1 + g, 256);  // every projection of the slot is read
            mx = fmaxf(xmax[g][0][row], xmax[g][1][row]);
            float M2 = mx * sl2e;
            float ls[4] = {0.0f, 0.0f, 0.0f, 0.0f};
            // P of this half into quarter 2 half (over half 0's scores, or
            // over half 0's projections, read before the barrier above)
            const uint32_t pc = 64u * half;
#pragma unroll
            for (int c = 0; c < 64; c += 32) {
                uint32_t pk16[16];
#pragma unroll
                for (int hh = 0; hh < 2; ++hh) {
                    uint32_t v[16];
                    tmem_ld16(so + kc0 + c + 16 * hh, v);
                    tmem_wait_ld();
#pragma unroll
                    for (int jj = 0; jj < 16; jj += 2) {
                        const float a0 = ex2_approx(
                            fmaf(__uint_as_float(v[jj]), sl2e, -M2));
                        const float a1 = ex2_approx(
                            fmaf(__uint_as_float(v[jj + 1]), sl2e, -M2));
                        ls[(jj >> 1) & 3] += a0 + a1;
                        pk16[8 * hh + (jj >> 1)] = pack_bf16x2(a0, a1);
                    }
                }
                tmem_st16(so + pc + (c >> 1), pk16);
            }
            float lsum = (ls[0] + ls[1]) + (ls[2] + ls[3]);
            xsum[g][half][row] = lsum;
            tc_fence_before();
            named_sync(1 + g, 256);  // every S read of the slot is done
            tc_fence_after();
            lsum = xsum[g][0][row] + xsum[g][1][row];
            float sp[32];
            uint32_t sp1[8];
            float dacc[4] = {0.0f, 0.0f, 0.0f, 0.0f};  // independent chains
            float denf = 0.0f;
            bool pass_fail = false;
#pragma unroll
            for (int ps = 1; ps < NP; ++ps) {
                // the previous pass's P goes to its P V product; this pass
                // scores the next 128 keys into columns [0, 128)
                tmem_wait_st();
                tc_fence_before();
                signal(&bars.p_full[g]);
                // the key buffer of pass ps - 1 is free since its scores
                // completed: the next block's keys, off the chain to the P V
                // product just handed over
                if (j + 1 < nblk && !gather_k(j + 1, ps - 1)) {
                    pass_fail = true;
                    break;
                }
                if (ps == 1) {
                    // per-bit factors of this half's tables (sp[0, 16):
                    // chunk half, sp[16, 32): chunk half + 2) and partial
                    // Den, while pass 0's P V product and pass 1's scores
                    // run. The A summary came by TMA: acquire its head's
                    // stage (complete already: the scores waited for it)
                    if ((j < 2 || blk_head(j) != blk_head(j - 2)) &&
                        !wwait(&bars.wb_full,
                               (blk_head(j) - blk_head(0)) & 1, 78)) {
                        pass_fail = true;
                        break;
                    }
                    race_factors16(pr, nt0 * G, beta, sp);
                    chunk_den<G, T>(sp, nt0, Asm + ta0 * R, dacc);
                    if (nt1 > 0) {
                        race_factors16(pr + 16, nt1 * G, beta, sp + 16);
                        chunk_den<G, T>(sp + 16, nt1, Asm + ta1 * R, dacc);
                        // the second chunk's factors wait for the P V
                        // product: kept as fp16 pairs (factors lie in
                        // (0.11, 0.89); relative rounding 2^-11, below the
                        // bf16 rounding of the features they make)
#pragma unroll
                        for (int q = 0; q < 8; ++q)
                            sp1[q] = pack_f16x2(sp[16 + 2 * q],
                                                sp[17 + 2 * q]);
                    }
                    xden[g][half][row] =
                        (dacc[0] + dacc[1]) + (dacc[2] + dacc[3]);
                }
                if (!wwait(&bars.s_full[g], (k * NP + ps) & 1, 79)) {
                    pass_fail = true;
                    break;
                }
                tc_fence_after();
                float mxb[4] = {-INFINITY, -INFINITY, -INFINITY, -INFINITY};
#pragma unroll
                for (int c = 0; c < 64; c += 16) {
                    uint32_t v[16];
                    tmem_ld16(so + pc + c, v);
                    tmem_wait_ld();
#pragma unroll
                    for (int jj = 0; jj < 16; ++jj)
                        mxb[jj & 3] = fmaxf(mxb[jj & 3], __uint_as_float(v[jj]));
                }
                xmax[g][half][row] =
                    fmaxf(fmaxf(mxb[0], mxb[1]), fmaxf(mxb[2], mxb[3]));
                named_sync(1 + g, 256);
                const float M2b =
                    fmaxf(xmax[g][0][row], xmax[g][1][row]) * sl2e;
                if (ps == 1)
                    denf = (xden[g][0][row] + xden[g][1][row]) *
                           (1.0f / (float)L);
                // online softmax: keep the running reference unless the
                // row's max grew by more than 2^8; then rescale the
                // accumulator (the previous P V product is complete: these
                // scores waited for it) and the running sum
                const bool need = M2b > M2 + 8.0f;
                const float f = need ? ex2_approx(M2 - M2b) : 1.0f;
                if (__any_sync(0xffffffffu, need)) {
#pragma unroll
                    for (int c = 0; c < 64; c += 16) {
                        uint32_t v[16];
                        tmem_ld16(so + nk + half * 64 + c, v);
                        tmem_wait_ld();
#pragma unroll
                        for (int q = 0; q < 16; ++q)
                            v[q] = __float_as_uint(__uint_as_float(v[q]) * f);
                        tmem_st16(so + nk + half * 64 + c, v);
                    }
                }
                if (need) {
                    lsum *= f;
                    M2 = M2b;
                }
                float lb[4] = {0.0f, 0.0f, 0.0f, 0.0f};
#pragma unroll
                for (int c = 0; c < 64; c += 32) {
                    uint32_t pk16[16];
#pragma unroll
                    for (int hh = 0; hh < 2; ++hh) {
                        uint32_t v[16];
                        tmem_ld16(so + pc + c + 16 * hh, v);
                        tmem_wait_ld();
#pragma unroll
                        for (int jj = 0; jj < 16; jj += 2) {
                            const float a0 = ex2_approx(
                                fmaf(__uint_as_float(v[jj]), sl2e, -M2));
                            const float a1 = ex2_approx(
                                fmaf(__uint_as_float(v[jj + 1]), sl2e, -M2));
                            lb[(jj >> 1) & 3] += a0 + a1;
                            pk16[8 * hh + (jj >> 1)] = pack_bf16x2(a0, a1);
                        }
                    }
                    tmem_st16(so + pc + (c >> 1), pk16);
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
            const float lam = lambda_tok ? lambda_tok[tok] : lambda;
            const float gs = gates ? gates[2 * tok] : 1.0f;
            const float gl = gates ? gates[2 * tok + 1] : 1.0f;
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
            signal(&bars.p_full[g]);
            // the last pass's key buffer and the query buffer are free since
            // the last scores completed: the next block's keys, the queries
            // of the block after next
            if ((j + 1 < nblk && !gather_k(j + 1, NP - 1)) ||
                (j + 2 < nblk && !gather_q(j + 2)))
                break;
            if (r > nk) {
                if (!wwait(&bars.pv_done[g], k & 1, 80)) break;
                tc_fence_after();
                if (nt1 > 0) {
                    float f1[16];
#pragma unroll
                    for (int q = 0; q < 8; ++q)
                        unpack_f16x2(sp1[q], f1[2 * q], f1[2 * q + 1]);
                    write_phi_chunk<G, T>(f1, nt1, ratio, so + cb1);
                }
                tmem_wait_st();
                tc_fence_before();
                signal(&bars.p2_full[g]);
            }
            if (!wwait(&bars.o_full[g], k & 1, 81)) break;
            tc_fence_after();
            // O = c1 acc, this half's 64 columns, straight from the
            // registers: fp32, or bf16 in 32-byte stores (a whole sector
            // each) when O is 32-byte aligned
            const bool o_a32 = ((uintptr_t)ox & 31u) == 0;
#pragma unroll
            for (int c = 0; c < 64; c += 16) {
                uint32_t v[16];
                tmem_ld16(so + nk + half * 64 + c, v);
                tmem_wait_ld();
                if constexpr (O32) {
                    float4 *dst = reinterpret_cast<float4 *>(
                        o32 + tok * (size_t)d + half * 64 + c);
#pragma unroll
                    for (int q = 0; q < 4; ++q)
                        dst[q] = make_float4(c1e * __uint_as_float(v[4 * q]),
                                             c1e * __uint_as_float(v[4 * q + 1]),
                                             c1e * __uint_as_float(v[4 * q + 2]),
                                             c1e * __uint_as_float(v[4 * q + 3]));
                } else {
                    uint32_t ob[8];
#pragma unroll
                    for (int q = 0; q < 8; ++q)
                        ob[q] = pack_bf16x2(c1e * __uint_as_float(v[2 * q]),
                                            c1e * __uint_as_float(v[2 * q + 1]));
                    uint16_t *dst = ox + tok * (size_t)d + half * 64 + c;
                    if (o_a32) {
                        st_global_v8(dst, ob);
                    } else {
                        uint4 *d4 = reinterpret_cast<uint4 *>(dst);
                        d4[0] = make_uint4(ob[0], ob[1], ob[2], ob[3]);
                        d4[1] = make_uint4(ob[4], ob[5], ob[6], ob[7]);
                    }
                }
            }
            tc_fence_before();
            signal(&bars.tmem_empty[g]);
            if (half == 0) {
                if (log_ds_out) log_ds_out[tok] = log_ds;
                if (dlr_out) dlr_out[tok] = denf;
                if (m_out) m_out[tok] = msp;
            }
        }
        cp_async_wait<0>();
    }
    tc_fence_before();
    __syncthreads();
    cluster_sync();  // no CTA leaves while the pair's MMAs may read it
    if (warp == kPrMmaWarp) tmem_dealloc_pair(tm, 512);
}

}  // namespace

bool pair_supported(const Plan &P) {
    const long rows = (long)P.N * P.BH;
    return tc_supported(P) && P.d == 128 && P.b == 256 && P.nb == 0 &&
           !P.sel && P.gamma == 4 && P.L <= 16 && P.N % 256 == 0 &&
           rows < (1L << 31);
}

size_t pair_smem(const Plan &P) {
    const size_t r = (size_t)P.r;
    return 1024 + 2 * (size_t)kPrNK * kPrD * 2 +
           (size_t)(kPrKRows0 + kPrKRows1) * kPrD * 2 + kPrNP * 16384 +
           (r * 128 + 1023) / 1024 * 1024 + (r * 4 + 1023) / 1024 * 1024;
}

cudaError_t launch_block_attn_pair(
    const Plan &P, const void *q, const void *k, const void *v,
    const uint16_t *w_bf16, const int32_t *perm_q, const int32_t *perm_k,
    const float *A, const uint16_t *Bh, const float *lambda_tok,
    const float *gates, void *o, float *log_d_sparse, float *d_lr,
    float *m_sparse, DeviceStatus *status, cudaStream_t st) {
    const size_t smem = pair_smem(P);
    const int bph = P.N / 256;
    const long total = (long)bph * P.BH;
    CUtensorMap tmW, tmB;
    cudaError_t e = make_tma_map_bf16(&tmW, w_bf16, (uint64_t)P.H * P.Lg_pad,
                                      P.d, 16u);
    if (e == cudaSuccess)
        e = make_tma_map_bf16(&tmB, Bh, (uint64_t)P.BH * P.r, P.d,
                              (uint32_t)P.r);
    if (e != cudaSuccess) return e;
    auto launch = [&](auto kern) {
        cudaError_t err = cudaFuncSetAttribute(
            kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
        if (err != cudaSuccess) return err;
        cudaLaunchConfig_t cfg = {};
        cudaLaunchAttribute attr[1];
        attr[0].id = cudaLaunchAttributeClusterDimension;
        attr[0].val.clusterDim.x = 2;
        attr[0].val.clusterDim.y = 1;
        attr[0].val.clusterDim.z = 1;
        cfg.blockDim = dim3(kPrThreads);
        cfg.dynamicSmemBytes = smem;
        cfg.stream = st;
        cfg.attrs = attr;
        cfg.numAttrs = 1;
        // one pair per two SMs that can hold it at once, at most one per
        // block
        int clusters = 0;
        cfg.gridDim = dim3(2 * 76);
        err = cudaOccupancyMaxActiveClusters(&clusters, kern, &cfg);
        if (err != cudaSuccess) return err;
        if (clusters < 1) return cudaErrorInvalidConfiguration;
        const long ncl = total < clusters ? total : clusters;
        cfg.gridDim = dim3((unsigned)(2 * ncl));
        return cudaLaunchKernelEx(
            &cfg, kern, (const uint16_t *)q, (const uint16_t *)k,
            (const uint16_t *)v, tmW, tmB, perm_q, perm_k, A, lambda_tok,
            gates, P.o32 ? nullptr : (uint16_t *)o,
            P.o32 ? (float *)o : nullptr, log_d_sparse, d_lr, m_sparse, P.N,
            P.H, P.L, P.Lg_pad, P.beta, P.eps, P.scale, P.lambda,
            P.fusion_mode, bph, total, status);
    };
    return P.o32 ? launch(k_block_attn_pair<true>)
                 : launch(k_block_attn_pair<false>);
}

}  // namespace elsaa
