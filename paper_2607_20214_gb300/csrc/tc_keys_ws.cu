// Warp-specialised RACE key side (Algorithm "RACE Low-Rank Attention
// Branch", steps 3-7) for bf16 inputs: one CTA accumulates the partial
// bucket summaries B += Phi_K^T V and A += Phi_K^T 1 of one chunk of keys of
// one head in tensor memory. A comes out of the same MMAs as B: the value
// tile is followed in shared memory by a panel of ones, so each MMA has
// N = d + 16 and its last 16 columns accumulate Phi^T 1.
//
// Roles (320 threads):
//   warp 0      loader (lane 0): TMA loads of key tiles (two buffers) and
//               value tiles (one buffer, one tile behind the keys);
//               completion is counted in bytes on the buffers' mbarriers.
//   warp 1      allocates tensor memory and issues the MMAs (lane 0): the
//               projections W^(l) K of tile i+1 (double-buffered in TMEM)
//               are issued before the summary MMAs of tile i.
//   warps 2-9   features: thread pairs (warps w, w + 4) share a key row and
//               split its tables (half h writes buckets of its tables into
//               the one shared feature tile). The tile is handed over per
//               half: a half may write tile i+1 as soon as the MMAs that
//               read its buckets of tile i are done.
// Every hand-off is an mbarrier with a bounded wait.
#include "device_common.cuh"
#include "tc_common.cuh"
#include "tc_race.cuh"

namespace elsaa {

namespace {

using namespace tc;

constexpr int kKwThreads = 320;

struct KwBars {
    uint64_t k_full[2], k_empty[2], v_full[2], v_empty[2], w_full, done;
    uint64_t proj_full[2];
    uint64_t phi_full[2], phi_empty[2];  // per row half
};

template <int G>
__global__ void __launch_bounds__(kKwThreads, 1)
    k_race_keys_ws(const __grid_constant__ CUtensorMap tmK,
                   const __grid_constant__ CUtensorMap tmV,
                   const __grid_constant__ CUtensorMap tmW, int N, int d,
                   int H,
                   int L, int r_pad, int Lg_pad, int chunk, float beta,
                   uint32_t tmem_cols, float *__restrict__ part,
                   DeviceStatus *status) {
    constexpr int R = 1 << G;
    extern __shared__ unsigned char smem_raw[];
    __shared__ KwBars bars;
    __shared__ uint32_t tbase;
    __shared__ int abort_flag;
    volatile int *abort = &abort_flag;
    const int s = blockIdx.x, bh = blockIdx.y, S = gridDim.x;
    const int h = bh % H;
    const int tid = threadIdx.x, warp = tid >> 5, lane_id = tid & 31;
    const int Lg = L * G, r = L * R;
    const int nM = r_pad >> 7;

    const uint32_t base = align1k(smem_u32(smem_raw));
    const uint32_t tileB = 128u * d * 2u;
    const uint32_t sW = base;
    const uint32_t sK0 = sW + align1k(Lg_pad * d * 2);  // two key tiles
    const uint32_t sV = sK0 + 2 * tileB;  // value tile, then a ones panel
    const uint32_t sPhi = sV + tileB + 16384u;  // one feature tile

    // TMEM columns: per M-tile an accumulator of d + 16 columns (B, then A
    // repeated 16 times), then two projection buffers of 64 columns.
    const uint32_t accN = (uint32_t)d + 16u;
    const uint32_t colP = nM * accN;

    if (warp == 1) tmem_alloc(&tbase, tmem_cols);
    if (tid == 0) {
        mbar_init(&bars.done, 1);
        mbar_init(&bars.w_full, 1);
        for (int b = 0; b < 2; ++b) {
            mbar_init(&bars.k_full[b], 1);
            mbar_init(&bars.k_empty[b], 1);
            mbar_init(&bars.v_full[b], 1);
            mbar_init(&bars.v_empty[b], 1);
            mbar_init(&bars.proj_full[b], 1);
            mbar_init(&bars.phi_full[b], 128);
            mbar_init(&bars.phi_empty[b], 1);
        }
        abort_flag = 0;
        fence_mbar_init();
    }
    for (int i = tid; i < 16384 / 16; i += kKwThreads)  // bf16 ones
        asm volatile("st.shared.v4.b32 [%0], {%1, %1, %1, %1};" ::"r"(
                         sV + tileB + i * 16),
                     "r"(0x3F803F80u)
                     : "memory");
    fence_proxy_async_smem();
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t t = tbase;
    // this head's bf16 planes (one TMA box of Lg_pad rows per 64 columns)
    if (tid == 0) {
        mbar_expect_tx(&bars.w_full, (uint32_t)Lg_pad * d * 2u);
        for (int pnl = 0; pnl < d / 64; ++pnl)
            tma_load_2d(sW + pnl * Lg_pad * 128, &tmW, 64 * pnl, h * Lg_pad,
                        &bars.w_full);
    }

    const int c0 = s * chunk;
    const int c1 = min(N, c0 + chunk);
    const int ntiles = c1 > c0 ? (c1 - c0 + 127) / 128 : 0;
    // buckets [0, sb) come from row half 0, [sb, r_pad) from half 1 (the
    // tail owner also zero-fills [r, r_pad)); M-tile m covers
    // [128 m, 128 m + 128)
    const int sb = table_split(L, G) * R;
    const bool h1_has = table_split(L, G) < L;
    auto tile_needs = [=](int m, int hf) {
        const int lo = 128 * m, hi = 128 * m + 128;
        if (hf == 0) return sb > lo || !h1_has;
        return h1_has && hi > sb;
    };
    auto last_mtile = [=](int hf) {  // last M-tile that reads half hf
        int last = -1;
        for (int m = 0; m < nM; ++m)
            if (tile_needs(m, hf)) last = m;
        return last;
    };

    if (warp == 0) {
        // ------------------------------------------------------------- loader
        if (lane_id == 0) {
            // K(i) needs the projection of tile i-2 done, V(i) the summary
            // MMAs of tile i-1; K runs ahead of V
            int iv = 0;
            for (int i = 0; i < ntiles; ++i) {
                const int b = i & 1;
                if (i >= 2 && !mbar_wait_or_abort(&bars.k_empty[b],
                                                  ((i >> 1) - 1) & 1, abort,
                                                  status, 61))
                    break;
                // rows past the chunk are loaded too (next head, or zeros
                // past the tensor) and get zero features
                const int y = bh * N + c0 + i * 128;
                mbar_expect_tx(&bars.k_full[b], tileB);
                for (int pnl = 0; pnl < d / 64; ++pnl)
                    tma_load_2d(sK0 + b * tileB + pnl * 16384, &tmK, 64 * pnl,
                                y, &bars.k_full[b]);
                // values up to tile i - 1 (one tile behind the keys)
                for (; iv < i; ++iv) {
                    if (iv >= 1 && !mbar_wait_or_abort(&bars.v_empty[0],
                                                       (iv - 1) & 1, abort,
                                                       status, 62))
                        break;
                    mbar_expect_tx(&bars.v_full[0], tileB);
                    for (int pnl = 0; pnl < d / 64; ++pnl)
                        tma_load_2d(sV + pnl * 16384, &tmV, 64 * pnl,
                                    bh * N + c0 + iv * 128, &bars.v_full[0]);
                }
            }
            for (; iv < ntiles; ++iv) {
                if (iv >= 1 && !mbar_wait_or_abort(&bars.v_empty[0],
                                                   (iv - 1) & 1, abort,
                                                   status, 62))
                    break;
                mbar_expect_tx(&bars.v_full[0], tileB);
                for (int pnl = 0; pnl < d / 64; ++pnl)
                    tma_load_2d(sV + pnl * 16384, &tmV, 64 * pnl,
                                bh * N + c0 + iv * 128, &bars.v_full[0]);
            }
        }
        __syncwarp();
    } else if (warp == 1) {
        // ----------------------------------------------------------- MMA issue
        if (lane_id == 0 && ntiles > 0) {
            const uint32_t id_proj = idesc_bf16(128, Lg_pad, false, false);
            const uint32_t id_b = idesc_bf16(128, d + 16, true, true);
            const int last0 = last_mtile(0), last1 = last_mtile(1);
            auto proj = [=](int it) {
                const uint32_t sK = sK0 + (it & 1) * tileB;
                const uint32_t dst = t + colP + 64u * (it & 1);
                for (int k = 0; k < d / 16; ++k) {
                    uint32_t oa = (k >> 2) * 128 * 128 + (k & 3) * 32;
                    uint32_t ow = (k >> 2) * Lg_pad * 128 + (k & 3) * 32;
                    mma_ss(dst, smem_desc(sK + oa, 16, 1024),
                           smem_desc(sW + ow, 16, 1024), id_proj, k > 0);
                }
                mma_commit(&bars.proj_full[it & 1]);
                mma_commit(&bars.k_empty[it & 1]);
            };
            // projections run two tiles ahead (both TMEM buffers); each
            // iteration issues the summary MMAs of tile i, then the
            // projection of tile i + 2
            bool ok = mbar_wait_or_abort(&bars.w_full, 0, abort, status, 60);
            for (int it = 0; it < 2 && it < ntiles && ok; ++it) {
                ok = mbar_wait_or_abort(&bars.k_full[it], 0, abort, status, 63);
                if (ok) {
                    tc_fence_after();
                    proj(it);
                }
            }
            for (int i = 0; i < ntiles && ok; ++i) {
                const int b = i & 1;
                ok = mbar_wait_or_abort(&bars.v_full[0], i & 1, abort,
                                        status, 66);
                bool got0 = false, got1 = false;
                for (int m = 0; m < nM && ok; ++m) {
                    if (tile_needs(m, 0) && !got0)
                        got0 = ok = mbar_wait_or_abort(&bars.phi_full[0], i & 1,
                                                       abort, status, 65);
                    if (ok && tile_needs(m, 1) && !got1)
                        got1 = ok = mbar_wait_or_abort(&bars.phi_full[1], i & 1,
                                                       abort, status, 65);
                    if (!ok) break;
                    tc_fence_after();
                    for (int k = 0; k < 8; ++k) {  // 128 keys, 16 per step
                        uint64_t a = smem_desc(sPhi + 2 * m * 16384 + k * 2048,
                                               16384, 1024);
                        uint32_t acc = (i > 0 || k > 0) ? 1u : 0u;
                        mma_ss(t + m * accN, a,
                               smem_desc(sV + k * 2048, 128 * 128, 1024), id_b,
                               acc);
                    }
                    if (m == last0) mma_commit(&bars.phi_empty[0]);
                    if (m == last1) mma_commit(&bars.phi_empty[1]);
                }
                if (!ok) break;
                mma_commit(&bars.v_empty[0]);
                if (i + 2 < ntiles) {
                    // the features of tile i have read projection buffer b
                    ok = mbar_wait_or_abort(&bars.k_full[b],
                                            ((i + 2) >> 1) & 1, abort, status,
                                            64);
                    if (!ok) break;
                    tc_fence_after();
                    proj(i + 2);
                }
            }
            if (ok) mma_commit(&bars.done);
        }
        __syncwarp();
    } else {
        // ------------------------------------------------------------ features
        const int cw = warp - 2;
        const int half = cw >> 2;
        const int row = (warp & 3) * 32 + lane_id;  // key row = TMEM lane
        const uint32_t lane = (uint32_t)((warp & 3) * 32) << 16;
        const int split = table_split(L, G);
        const int l0 = half ? split : 0, l1 = half ? L : split;
        const bool tail_owner = (l1 == L) && (l1 > l0 || half == 0);
        auto wwait = [=](uint64_t *bar, uint32_t par, int site) {
            return __all_sync(0xffffffffu,
                              mbar_wait_or_abort(bar, par, abort, status,
                                                 site));
        };
        bool ok = true;
        const bool writes = l1 > l0 || tail_owner;  // this half has buckets
        const int hb = (l1 > l0 || half == 0) ? half : 0;  // barrier to use
        for (int i = 0; i < ntiles; ++i) {
            const int b = i & 1;
            ok = wwait(&bars.proj_full[b], (i >> 1) & 1, 67);
            if (ok && i >= 1 && writes)
                ok = wwait(&bars.phi_empty[hb], (i - 1) & 1, 68);
            if (!ok) break;
            tc_fence_after();
            float sp[32];
            race_bits32(t + lane + colP + 64u * b + l0 * G, (l1 - l0) * G,
                        beta, sp);
            const bool valid = c0 + i * 128 + row < c1;
            float buf[8];
#pragma unroll
            for (int lt = 0; lt < 32 / G; ++lt) {
                if (G == 4 && l0 + lt < l1) {
                    float u[4], w[4];
                    table_uw4(&sp[lt * G], valid ? 1.0f : 0.0f, u, w);
                    uint32_t pk[8];
                    table_pack4(u, w, pk);
                    const int cc = (l0 * R + lt * R) >> 3;
#pragma unroll
                    for (int hh = 0; hh < 2; ++hh)
                        asm volatile(
                            "st.shared.v4.b32 [%0], {%1, %2, %3, %4};" ::"r"(
                                sPhi + panel_offset(row, cc + hh, 128)),
                            "r"(pk[4 * hh]), "r"(pk[4 * hh + 1]),
                            "r"(pk[4 * hh + 2]), "r"(pk[4 * hh + 3])
                            : "memory");
                } else if (l0 + lt < l1) {
                    float phi[R];
                    table_phi<G>(&sp[lt * G], phi);
#pragma unroll
                    for (int q = 0; q < R; ++q) {
                        const int prel = lt * R + q;  // l0 * R is 32-aligned
                        buf[prel & 7] = valid ? phi[q] : 0.0f;
                        if ((prel & 7) == 7)
                            st_shared_bf16x8(
                                sPhi + panel_offset(row, (l0 * R + prel) >> 3,
                                                    128),
                                buf);
                    }
                }
            }
            if (tail_owner) {
                if ((r & 7) != 0) {  // partial last chunk (< 8 buckets)
                    for (int q = r & 7; q < 8; ++q) buf[q] = 0.0f;
                    st_shared_bf16x8(sPhi + panel_offset(row, r >> 3, 128),
                                     buf);
                }
                for (int c = (r + 7) >> 3; c < (r_pad >> 3); ++c)
                    st_shared_zero16(sPhi + panel_offset(row, c, 128));
            }
            fence_proxy_async_smem();
            tc_fence_before();
            mbar_arrive(&bars.phi_full[half]);
        }
        // partial summaries of this chunk (each half: half the columns)
        float *out = part + ((size_t)bh * S + s) * ((size_t)r * d + r);
        if (ok && ntiles > 0) ok = wwait(&bars.done, 0, 69);
        if (ok && ntiles > 0) {
            tc_fence_after();
            for (int m = 0; m < nM; ++m) {
                const int rrow = m * 128 + row;
                for (int c = half * (d >> 1); c < (half + 1) * (d >> 1);
                     c += 32) {
                    uint32_t v[32];
                    tmem_ld32(t + lane + m * accN + c, v);
                    tmem_wait_ld();
                    if (rrow < r) {
                        float4 *dst = reinterpret_cast<float4 *>(
                            out + (size_t)rrow * d + c);
#pragma unroll
                        for (int j = 0; j < 8; ++j)
                            dst[j] = make_float4(
                                __uint_as_float(v[4 * j]),
                                __uint_as_float(v[4 * j + 1]),
                                __uint_as_float(v[4 * j + 2]),
                                __uint_as_float(v[4 * j + 3]));
                    }
                }
                if (half == 0) {
                    uint32_t a16[16];
                    tmem_ld16(t + lane + m * accN + d, a16);
                    tmem_wait_ld();
                    if (rrow < r)
                        out[(size_t)r * d + rrow] = __uint_as_float(a16[0]);
                }
            }
        } else if (ntiles == 0) {
            for (int i = tid - 64; i < r * d + r; i += 256) out[i] = 0.0f;
        }
    }
    tc_fence_before();
    __syncthreads();
    if (warp == 1) tmem_dealloc(t, tmem_cols);
}

uint32_t pow2_cols_kw(uint32_t n) {
    uint32_t c = 32;
    while (c < n) c <<= 1;
    return c;
}

}  // namespace

size_t race_keys_ws_smem(const Plan &P) {
    const size_t r_pad = (P.r + 127) / 128 * 128;
    const size_t lg_pad = (P.L * P.gamma + 15) / 16 * 16;
    return 1024 + (lg_pad * P.d * 2 + 1023) / 1024 * 1024 +
           3 * (size_t)128 * P.d * 2 + 16384 + 128 * r_pad * 2;
}

uint32_t race_keys_ws_cols(const Plan &P) {
    const int r_pad = (P.r + 127) / 128 * 128;
    return pow2_cols_kw((r_pad / 128) * (P.d + 16) + 128);
}

namespace {
__global__ void k_prep_planes(const float *__restrict__ w, int H, int Lg,
                              int Lg_pad, int d, uint16_t *__restrict__ out) {
    const long n = (long)H * Lg_pad * d;
    for (long i = blockIdx.x * (long)blockDim.x + threadIdx.x; i < n;
         i += (long)gridDim.x * blockDim.x) {
        const int c = (int)(i % d);
        const long hr = i / d;
        const int row = (int)(hr % Lg_pad), h = (int)(hr / Lg_pad);
        const float x = row < Lg ? w[((long)h * Lg + row) * d + c] : 0.0f;
        const __nv_bfloat16 b = __float2bfloat16_rn(x);
        out[i] = *reinterpret_cast<const uint16_t *>(&b);
    }
}
}  // namespace

cudaError_t launch_prep_planes(const Plan &P, const float *w_race,
                               uint16_t *w_bf16, cudaStream_t st) {
    const long n = (long)P.H * P.Lg_pad * P.d;
    const int blocks = (int)((n + 255) / 256 < 1024 ? (n + 255) / 256 : 1024);
    k_prep_planes<<<blocks, 256, 0, st>>>(w_race, P.H, P.L * P.gamma,
                                          P.Lg_pad, P.d, w_bf16);
    return cudaGetLastError();
}

cudaError_t launch_race_keys_ws(const Plan &P, const void *k, const void *v,
                                const uint16_t *w_bf16, float *part,
                                DeviceStatus *status, cudaStream_t st) {
    const int r_pad = (P.r + 127) / 128 * 128;
    const int lg_pad = (P.L * P.gamma + 15) / 16 * 16;
    const uint32_t cols = race_keys_ws_cols(P);
    const size_t need = race_keys_ws_smem(P);
    // cap residency at what TMEM allows
    const int fit = 512 / (int)cols;
    const size_t cap = (size_t)233472 / (fit + 1) + 1;
    const size_t smem = need > cap ? need : cap;
    dim3 grid(P.S, P.BH);
    CUtensorMap tmK, tmV, tmW;
    const uint64_t rows = (uint64_t)P.BH * P.N;
    cudaError_t e = make_tma_map_bf16(&tmK, k, rows, P.d, 128);
    if (e == cudaSuccess) e = make_tma_map_bf16(&tmV, v, rows, P.d, 128);
    if (e == cudaSuccess)
        e = make_tma_map_bf16(&tmW, w_bf16, (uint64_t)P.H * P.Lg_pad, P.d,
                              (uint32_t)P.Lg_pad);
    if (e != cudaSuccess) return e;
    auto launch = [&](auto kern) {
        cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             (int)smem);
        kern<<<grid, kKwThreads, smem, st>>>(
            tmK, tmV, tmW, P.N, P.d, P.H, P.L, r_pad, lg_pad, P.chunk,
            P.beta, cols, part, status);
        return cudaGetLastError();
    };
    switch (P.gamma) {
        case 1: return launch(k_race_keys_ws<1>);
        case 2: return launch(k_race_keys_ws<2>);
        case 3: return launch(k_race_keys_ws<3>);
        case 4: return launch(k_race_keys_ws<4>);
        case 5: return launch(k_race_keys_ws<5>);
        case 6: return launch(k_race_keys_ws<6>);
        default: return cudaErrorInvalidValue;
    }
}

}  // namespace elsaa
