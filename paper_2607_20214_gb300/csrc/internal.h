// Internal declarations shared by the CUDA translation units of libelsaa.
// Nothing here is part of the public ABI (see include/elsaa.h).
#pragma once

#include <cuda.h>
#include <cuda_runtime.h>
#include <stddef.h>
#include <stdint.h>

#include "../../include/elsaa.h"

namespace elsaa {

// Tokens per hash tile: one CTA hashes, histograms and locally ranks one tile.
constexpr int kHashTile = 128;
// Queries per CTA of the CUDA-core block-attention kernel.
constexpr int kSimtQT = 32;
// Buckets per slice in the CUDA-core RACE kernels.
constexpr int kSliceBuckets = 64;

// In-band device status (first bytes of the workspace). code == 0: no fault.
struct DeviceStatus {
    int code;
    int where;
    int info0;
    int info1;
};
// Status codes written by kernels (first writer wins).
constexpr int kDevSortRange = 1;     // a scatter position fell outside [0, N)
constexpr int kDevPermRange = 2;     // a permutation entry fell outside [0, N)
constexpr int kDevWaitTimeout = 3;   // a bounded mbarrier wait ran out
constexpr int kDevTmem = 4;          // tensor-memory allocation failed

// The CTA (of `grid` over `total` work items, CTA c taking items
// [total c / grid, total (c + 1) / grid)) that works on item t.
__host__ __device__ inline long range_owner(long t, long total, long grid) {
    return ((t + 1) * grid + total - 1) / total - 1;
}

// Resolved problem geometry and workspace layout (all offsets in bytes).
struct Plan {
    int B, H, N, d, BH;
    int dtype;
    int b;           // block size
    int n_s, bins;   // sort bits, 2^n_s
    int gray;
    int L, gamma, R, r;  // tables, bits, buckets per table, total buckets
    int tables_per_slice, slices;
    int S, chunk;    // RACE key chunks per head and tokens per chunk
    int tiles;       // hash tiles per head
    float beta, eps, scale, lambda;
    int fusion_mode;
    int nb;          // neighbouring sorted key blocks on each side
    int impl;        // resolved: 1 = SIMT, 2 = tensor core
    int Lg_pad;      // L * gamma rounded up to 16 (projection MMA width)
    int o32;         // write O as fp32 although the inputs are bf16
    int sel;         // 0: sorted blocks; 1: per-query top-k selector
    int tk_k, tk_c;  // top-k: keys per query, candidate blocks per block
    size_t off_status, off_keyrank, off_hist, off_perm, off_part, off_A,
        off_B, off_Bh, off_W, off_sums, off_cand, off_mask, total;
};

// Records a one-line error for elsaa_last_error() and returns `code`.
int set_last_error(int code, const char *fmt, ...);

// Fills `plan` from validated parameters. Returns ELSAA_OK or an error code
// and message (no CUDA calls).
int make_plan(const elsaa_params *p, Plan *plan, const char **msg);

// Launchers (return cudaError_t of the launch). Pointers are device pointers.
cudaError_t launch_sort_hash(const Plan &P, const void *q, const void *k,
                             const float *w_sort, uint32_t *keyrank,
                             int *hist, DeviceStatus *status,
                             cudaStream_t st);
cudaError_t launch_sort_scan(const Plan &P, int *hist, cudaStream_t st);
cudaError_t launch_sort_scatter(const Plan &P, const uint32_t *keyrank,
                                const int *hist, int32_t *perm_q,
                                int32_t *perm_k, DeviceStatus *status,
                                cudaStream_t st);
cudaError_t launch_race_partial_simt(const Plan &P, const void *k,
                                     const void *v, const float *w_race,
                                     float *part, cudaStream_t st);
// k_race_partial with fp32 values and per-token A weights (backward pass:
// gB = sum phi(x_i) vals_i^T, gA = sum phi(x_i) wA_i).
cudaError_t launch_race_partial_weighted(const Plan &P, const void *x,
                                         const float *vals, const float *wA,
                                         const float *w_race, float *part,
                                         cudaStream_t st);
cudaError_t launch_race_reduce(const Plan &P, const float *part, float *A,
                               float *Bm, uint16_t *Bh, cudaStream_t st);
cudaError_t launch_block_attn_simt(
    const Plan &P, const void *q, const void *k, const void *v,
    const float *w_race, const int32_t *perm_q, const int32_t *perm_k,
    const float *A, const float *Bm, const float *lambda_tok,
    const float *gates, void *o, float *log_d_sparse, float *d_lr,
    float *m_sparse, DeviceStatus *status, cudaStream_t st,
    const int32_t *cand = nullptr, const uint32_t *selmask = nullptr);

// The gate network run inside elsaa_forward_gated (gates.cu kernels):
// its description, the bf16 operand image it writes, and its outputs.
struct GateFusion {
    const elsaa_gate_mlp *mlp;
    uint16_t *gate_ws;  // launch_gates' bf16 operand image
    float *gates, *lam;
};

// Per-query top-k selector (topk.cu).
bool topk_supported(const Plan &P, const char **msg);
// stage 0: block sums; 1: candidate blocks; 2: per-query selection
cudaError_t launch_topk(int stage, const Plan &P, const void *q,
                        const void *k, const int32_t *perm_q,
                        const int32_t *perm_k, float *sums, int32_t *cand,
                        uint32_t *selmask, DeviceStatus *status,
                        cudaStream_t st);
cudaError_t launch_topk_export(const Plan &P, const int32_t *perm_q,
                               const int32_t *perm_k, const int32_t *cand,
                               const uint32_t *selmask, int32_t *out,
                               DeviceStatus *status, cudaStream_t st);

// Tensor-core (tcgen05) path for bf16 inputs.
bool tc_supported(const Plan &P);
// Chunks per head of the tensor-core RACE key kernel; writes tokens per chunk.
int tc_race_chunks(const Plan &P, int *chunk);


// Backward pass (bwd.cu), CUDA cores.
size_t bwd_block_smem(const Plan &P);
size_t bwd_keys_smem(const Plan &P);
bool bwd_supported(const Plan &P);
cudaError_t launch_bwd_block(const Plan &P, const void *q, const void *k,
                             const void *v, const void *d_o,
                             const float *w_race, const float *A,
                             const float *Bm, const int32_t *perm_q,
                             const int32_t *perm_k, const float *lambda_tok,
                             const float *gates, float *dq, float *dk,
                             float *dv, float *d_gates, float *d_lambda,
                             float *gnum, float *gden, DeviceStatus *status,
                             cudaStream_t st);
cudaError_t launch_bwd_keys(const Plan &P, const void *k, const void *v,
                            const float *w_race, const float *gA,
                            const float *gB, float *dk, float *dv,
                            cudaStream_t st);

// Tensor-core backward (bwd_tc.cu): the block kernel also sums gB, gA per
// head into bwd_tc_segments(P) partials per head (layout of the RACE chunk
// partials), which the key-side kernel adds up when it starts on a head.
bool bwd_tc_supported(const Plan &P);
size_t bwd_tc_smem(const Plan &P);
int bwd_tc_grid(const Plan &P);
// bf16 copy (round to nearest even) of n fp32 values.
cudaError_t launch_bf16_image(const float *x, uint16_t *y, size_t n,
                              cudaStream_t st);
// launch_prep_planes and launch_bf16_image in one launch (n a multiple of
// 4, x 16-byte and y 8-byte aligned; cudaErrorInvalidValue otherwise).
cudaError_t launch_planes_and_image(const Plan &P, const float *w_race,
                                    uint16_t *w_bf16, const float *x,
                                    uint16_t *y, size_t n, cudaStream_t st);
int bwd_tc_segments(const Plan &P);
cudaError_t launch_bwd_block_tc(const Plan &P, const void *q, const void *k,
                                const void *v, const void *d_o,
                                const uint16_t *w_bf16, const uint16_t *Bh,
                                const float *A, const int32_t *perm_q,
                                const int32_t *perm_k, const float *lambda_tok,
                                const float *gates, float *dq, float *dk,
                                float *dv, float *d_gates, float *d_lambda,
                                float *part, DeviceStatus *status,
                                cudaStream_t st);

size_t bwd_keys_tc_smem(const Plan &P);
cudaError_t launch_bwd_keys_tc(const Plan &P, const void *k, const void *v,
                               const uint16_t *w_bf16, const float *part,
                               float *dk, float *dv, DeviceStatus *status,
                               cudaStream_t st);

// Causal variant (causal.cu).
bool causal_tc_supported(const Plan &P, int n_leaf);
cudaError_t launch_seg_sort(const Plan &P, int Lv, const uint32_t *keyrank,
                            int32_t *perms, cudaStream_t st);
cudaError_t launch_causal_attn(const Plan &P, int mode, int n_leaf, int level,
                               const void *q, const void *k, const void *v,
                               const int32_t *perms, int *next_item, float *RO,
                               float *RL, DeviceStatus *status,
                               cudaStream_t st);
int causal_segments(const Plan &P);
cudaError_t launch_causal_scan(const Plan &P, const void *k, const void *v,
                               const uint16_t *w_bf16, float *part,
                               uint16_t *sBh, float *sA, DeviceStatus *status,
                               cudaStream_t st);
cudaError_t launch_causal_race(const Plan &P, const void *q, const void *k,
                               const void *v, const uint16_t *w_bf16,
                               const uint16_t *sBh, const float *sA,
                               const float *RO, const float *RL,
                               const float *lambda_tok, const float *gates,
                               void *o, float *log_ds, float *dlr, float *m,
                               DeviceStatus *status, cudaStream_t st);

// One bounded mbarrier wait that can never complete (selftest.cu).
cudaError_t launch_selftest_wait(DeviceStatus *status, int limit_ms,
                                 cudaStream_t st);

// Token-wise gate MLP and query-dependent lambda (gates.cu).
int gate_ng(int hidden);
bool gate_tc_supported(const Plan &P);
size_t gate_workspace_bytes(const Plan &P, int hidden);
cudaError_t launch_gates(const Plan &P, const elsaa_gate_mlp &m,
                         const void *q, float *gates, float *lam_out,
                         uint16_t *w_bf16, DeviceStatus *status,
                         cudaStream_t st);

// Row-major bf16 matrix [rows x cols] as a TMA tensor map with boxes of
// 64 columns x box_rows rows and 128-byte swizzle (the panel layout).
// Returns cudaSuccess or an error if the driver entry point is missing or
// the encoding is rejected.
cudaError_t make_tma_map_bf16(CUtensorMap *map, const void *base,
                              uint64_t rows, uint64_t cols, uint32_t box_rows);
// Row-major fp32 matrix [rows x cols] with boxes of box_cols = 32 columns
// (128 bytes) x box_rows rows and 128-byte swizzle: the 16-byte chunk c of
// box row j lands at chunk c ^ (j mod 8).
cudaError_t make_tma_map_f32(CUtensorMap *map, const void *base,
                             uint64_t rows, uint64_t cols, uint32_t box_cols,
                             uint32_t box_rows);
// The same (bf16) with boxes of box_cols = 16, 32 or 64 columns (32, 64 or 128
// bytes per row) and the swizzle of that width (32, 64 or 128 bytes): the
// 16-byte chunk c of box row r lands at chunk c ^ ((r / (8 / (box_cols / 8)))
// mod (box_cols / 8)).
cudaError_t make_tma_map_bf16_narrow(CUtensorMap *map, const void *base,
                                     uint64_t rows, uint64_t cols,
                                     uint32_t box_cols, uint32_t box_rows);

// RACE planes as bf16 rows [H][Lg_pad][d] (rows >= L * gamma zero), the
// operand image the tensor-core kernels load with TMA.
cudaError_t launch_prep_planes(const Plan &P, const float *w_race,
                               uint16_t *w_bf16, cudaStream_t st);

// Warp-specialised RACE key summaries (tensor-core path).
size_t race_keys_ws_smem(const Plan &P);
uint32_t race_keys_ws_cols(const Plan &P);
cudaError_t launch_race_keys_ws(const Plan &P, const void *k, const void *v,
                                const uint16_t *w_bf16, float *part,
                                DeviceStatus *status, cudaStream_t st);

// Persistent warp-specialised block attention (key blocks of <= 128).
bool ws_supported(const Plan &P);
cudaError_t launch_block_attn_ws(
    const Plan &P, const void *q, const void *k, const void *v,
    const uint16_t *w_bf16, const int32_t *perm_q, const int32_t *perm_k,
    const float *A, const uint16_t *Bh, const float *lambda_tok,
    const float *gates, void *o, float *log_d_sparse, float *d_lr,
    float *m_sparse, DeviceStatus *status, cudaStream_t st,
    const int32_t *cand = nullptr, const uint32_t *selmask = nullptr);

// Block attention for key blocks of 256 on CTA pairs (cta_group::2 MMAs):
// bf16, d_h = 128, gamma = 4, no neighbours or selector, N a multiple of 256.
bool pair_supported(const Plan &P);
size_t pair_smem(const Plan &P);
cudaError_t launch_block_attn_pair(
    const Plan &P, const void *q, const void *k, const void *v,
    const uint16_t *w_bf16, const int32_t *perm_q, const int32_t *perm_k,
    const float *A, const uint16_t *Bh, const float *lambda_tok,
    const float *gates, void *o, float *log_d_sparse, float *d_lr,
    float *m_sparse, DeviceStatus *status, cudaStream_t st);

}  // namespace elsaa
