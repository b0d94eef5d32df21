// RACE feature helpers shared by the tensor-core kernels (tc.cu, tc_ws.cu).
#pragma once

#include "device_common.cuh"
#include "tc_common.cuh"

namespace elsaa {
namespace tc {

constexpr float kLog2e = 1.4426950408889634f;
constexpr float kLn2 = 0.6931471805599453f;

__device__ __forceinline__ uint32_t align1k(uint32_t x) {
    return (x + 1023u) & ~1023u;
}

// RACE planes of one head as bf16 rows [Lg_pad x d] in the panel layout;
// rows >= Lg are zero.
// With row0 / prows: the planes are rows [row0, row0 + Lg_pad) of a panel
// layout of prows rows (planes stacked under a key tile).
__device__ inline void load_planes_bf16(uint32_t dst, const float *w, int Lg,
                                 int Lg_pad, int d, int tid, int nthreads,
                                 int row0 = 0, int prows = 0) {
    const int chunks = d >> 3;
    if (prows == 0) prows = Lg_pad;
    for (int i = tid; i < Lg_pad * chunks; i += nthreads) {
        int row = i / chunks, c = i - row * chunks;
        uint32_t addr = dst + panel_offset(row0 + row, c, prows);
        if (row < Lg) {
            const float4 *src =
                reinterpret_cast<const float4 *>(w + (size_t)row * d + c * 8);
            float4 a = src[0], b = src[1];
            float v[8] = {a.x, a.y, a.z, a.w, b.x, b.y, b.z, b.w};
            st_shared_bf16x8(addr, v);
        } else {
            st_shared_zero16(addr);
        }
    }
}

// Two threads share each row (warps w and w + 4 read the same TMEM lanes).
// The RACE tables of a row are split between them at table `split`, chosen
// so that each half's buckets start on a 32-bucket boundary (whole TMEM
// store groups) and each half reads at most 32 projection columns.
__host__ __device__ inline int table_split(int L, int G) {
    const int R = 1 << G;
    const int unit = R >= 32 ? 1 : 32 / R;  // tables per 32 buckets
    int split = ((L + 1) / 2 + unit - 1) / unit * unit;
    return split > L ? L : split;
}

// Per-bit factors sp[j] = sigmoid(2 beta tanh(a_j)) of the projection
// columns [col0, col0 + 32) of this thread's TMEM lane; entries past `ncols`
// are set to 1/2 and not used.
__device__ __forceinline__ void race_bits32(uint32_t taddr, int ncols,
                                           float beta, float (&sp)[32]) {
    uint32_t pr[32];
    tmem_ld32(taddr, pr);
    tmem_wait_ld();
#pragma unroll
    for (int j = 0; j < 32; ++j) {
        if (j < ncols) {
            float t = tanh_approx(beta * tanh_approx(__uint_as_float(pr[j])));
            sp[j] = fmaf(0.5f, t, 0.5f);  // 1/2 + tanh(beta u)/2
        } else {
            sp[j] = 0.5f;
        }
    }
}

// The per-bit factors of 16 projections already loaded from TMEM (fp32
// bits in pr): sp[j] for j < 16, entries past `ncols` set to 1/2.
__device__ __forceinline__ void race_factors16(const uint32_t *pr, int ncols,
                                               float beta, float *sp) {
#pragma unroll
    for (int j = 0; j < 16; ++j) {
        if (j < ncols) {
            float t = tanh_approx(beta * tanh_approx(__uint_as_float(pr[j])));
            sp[j] = fmaf(0.5f, t, 0.5f);
        } else {
            sp[j] = 0.5f;
        }
    }
}

// race_bits32 over 16 projection columns: sp[j] for j < 16, entries past
// `ncols` set to 1/2. The TMEM load is waited for inside.
__device__ __forceinline__ void race_bits16(uint32_t taddr, int ncols,
                                           float beta, float *sp) {
    uint32_t pr[16];
    tmem_ld16(taddr, pr);
    tmem_wait_ld();
    race_factors16(pr, ncols, beta, sp);
}

// Features of table l from its G per-bit factors: phi[r] = prod_b (bit b of
// r ? sp[b] : 1 - sp[b]), r < 2^G.
template <int G>
__device__ __forceinline__ void table_phi(const float *sp, float *phi,
                                          float init = 1.0f) {
    phi[0] = init;  // a common factor of the whole table (1 or a scale)
#pragma unroll
    for (int b = 0; b < G; ++b) {
        const float p = sp[b], q = 1.0f - p;
#pragma unroll
        for (int r = 0; r < (1 << b); ++r) {
            phi[r + (1 << b)] = phi[r] * p;
            phi[r] *= q;
        }
    }
}


// gamma = 4: the 16 features of one table factor as an outer product,
// phi[i + 4 j] = u[i] * w[j], with u over hash bits 0-1 and w over bits 2-3:
// u = (q0 q1, p0 q1, q0 p1, p0 p1), w = (q2 q3, p2 q3, q2 p3, p2 p3),
// p_b = sp[b], q_b = 1 - p_b. `scale` multiplies every feature.
__device__ __forceinline__ void table_uw4(const float *sp, float scale,
                                          float (&u)[4], float (&w)[4]) {
    const float p0 = sp[0], q0 = 1.0f - p0, p1 = sp[1], q1 = 1.0f - p1;
    const float p2 = sp[2], q2 = 1.0f - p2, p3 = sp[3], q3 = 1.0f - p3;
    const float a = q1 * scale, c = p1 * scale;
    u[0] = q0 * a;
    u[1] = p0 * a;
    u[2] = q0 * c;
    u[3] = p0 * c;
    w[0] = q2 * q3;
    w[1] = p2 * q3;
    w[2] = q2 * p3;
    w[3] = p2 * p3;
}

// sum_r phi_r A_r of one gamma = 4 table = sum_j w_j (u . A[4 j .. 4 j + 3]);
// A: 16 floats in shared memory, 16-byte aligned.
__device__ __forceinline__ float table_dot4(const float (&u)[4],
                                            const float (&w)[4],
                                            const float *A) {
    float acc[4];
#pragma unroll
    for (int j = 0; j < 4; ++j) {
        const float4 a = *reinterpret_cast<const float4 *>(A + 4 * j);
        acc[j] = fmaf(u[3], a.w, fmaf(u[2], a.z, fmaf(u[1], a.y, u[0] * a.x)));
    }
    return fmaf(w[3], acc[3], fmaf(w[2], acc[2], fmaf(w[1], acc[1], w[0] * acc[0])));
}

// Packed bf16 features of one gamma = 4 table: out[k] holds buckets
// (2k, 2k + 1), k < 8.
__device__ __forceinline__ void table_pack4(const float (&u)[4],
                                            const float (&w)[4],
                                            uint32_t *out) {
#pragma unroll
    for (int j = 0; j < 4; ++j) {
        out[2 * j] = pack_bf16x2(u[0] * w[j], u[1] * w[j]);
        out[2 * j + 1] = pack_bf16x2(u[2] * w[j], u[3] * w[j]);
    }
}

// Writes the pre-scaled features phi * scale of tables [l0, l1) of this
// thread's query row, for buckets [lo, hi), as packed bf16 pairs into TMEM
// with bucket lo at `taddr`. l0 * R and lo are multiples of 32 and hi of 16;
// buckets go out in groups of 32 (16 columns), the last half group padded
// with zeros.
template <int G>
__device__ __forceinline__ void write_phi_tmem(const float (&sp)[32], int l0,
                                               int l1, int r, float scale,
                                               int lo, int hi,
                                               uint32_t taddr) {
    constexpr int R = 1 << G;
    uint32_t buf[16];
#pragma unroll
    for (int lt = 0; lt < 32 / G; ++lt) {
        if (l0 + lt < l1) {
            float phi[R];
            table_phi<G>(&sp[lt * G], phi, scale);
#pragma unroll
            for (int q = 0; q < R; q += 2) {
                const int prel = lt * R + q;     // even, relative to l0 * R
                const int slot = (prel >> 1) & 15;
                buf[slot] = pack_bf16x2(phi[q], phi[q + 1]);
                const int p = l0 * R + prel;      // absolute bucket
                const bool last = p + 2 == r;
                if (slot == 15 || last) {
                    if (last) {
#pragma unroll
                        for (int z = 0; z < 16; ++z)
                            if (z > slot) buf[z] = 0u;
                    }
                    const int g = p - 2 * slot;  // first bucket of the group
                    if (g >= lo && g < hi)
                        tmem_st16(taddr + ((g - lo) >> 1), buf);
                }
            }
        }
    }
}

// sum over tables t < nt of phi_t . A_t for the tables of one 64-bucket
// chunk (at most TT of them; per-bit factors sp[t * G ..], A of the chunk's
// first table at A). Four independent partial sums in acc.
template <int G, int TT>
__device__ __forceinline__ void chunk_den(const float *sp, int nt,
                                          const float *A, float (&acc)[4]) {
    constexpr int R = 1 << G;
#pragma unroll
    for (int t = 0; t < TT; ++t) {
        if (t < nt) {
            if constexpr (G == 4) {
                float u[4], w[4];
                table_uw4(&sp[t * G], 1.0f, u, w);
                acc[t & 3] += table_dot4(u, w, A + t * R);
            } else {
                float phi[R];
                table_phi<G>(&sp[t * G], phi);
#pragma unroll
                for (int q = 0; q < R; ++q)
                    acc[q & 3] = fmaf(phi[q], A[t * R + q], acc[q & 3]);
            }
        }
    }
}

// Writes the features phi * scale of the nt (<= TT) tables of one 64-bucket
// chunk as packed bf16 pairs into TMEM: bucket pair (2k, 2k + 1) of the
// chunk at column taddr + k, k < 32, in two stores of 16 columns (the second
// only when the chunk holds more than 32 buckets). Pairs past the chunk's
// last table are zero.
template <int G, int TT>
__device__ __forceinline__ void write_phi_chunk(const float *sp, int nt,
                                                float scale, uint32_t taddr) {
    constexpr int R = 1 << G;
    static_assert(TT * R == 64, "a chunk is 64 buckets");
    uint32_t buf[16];
#pragma unroll
    for (int t = 0; t < TT; ++t) {
        uint32_t pk[R / 2];
        if (t < nt) {
            if constexpr (G == 4) {
                float u[4], w[4];
                table_uw4(&sp[t * G], scale, u, w);
                table_pack4(u, w, pk);
            } else {
                float phi[R];
                table_phi<G>(&sp[t * G], phi, scale);
#pragma unroll
                for (int q = 0; q < R; q += 2)
                    pk[q >> 1] = pack_bf16x2(phi[q], phi[q + 1]);
            }
        } else {
#pragma unroll
            for (int q = 0; q < R / 2; ++q) pk[q] = 0u;
        }
#pragma unroll
        for (int q = 0; q < R / 2; ++q) {
            const int k = t * (R / 2) + q;
            buf[k & 15] = pk[q];
            if ((k & 15) == 15 && (k < 16 || nt * R > 32))
                tmem_st16(taddr + (uint32_t)(k - 15), buf);
        }
    }
}

// TMEM column of K-step k (16 keys or buckets = 8 packed bf16 columns) of
// the quarter pair starting at col0: quarters (col0, col0 + 64) of 32
// columns each, the A operand of the P V and Phi'B products in the block
// kernels' slots.
__device__ __forceinline__ uint32_t quarter_col(int k, int col0) {
    return (uint32_t)(col0 + (k < 4 ? 8 * k : 64 + 8 * (k - 4)));
}

}  // namespace tc
}  // namespace elsaa
