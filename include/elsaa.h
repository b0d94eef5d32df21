/*
 * elsaa.h - C ABI of the GB300 (sm_103a) ELSAA attention operator.
 *
 * ELSAA (Efficient Low-rank and Sparse Approximation of Attention) replaces
 * dense attention after the Q/K/V projections by two branches and a fusion:
 *   - the sortLSH sparse branch (Section 3.2; Algorithm "sortLSH Sparse Exact
 *     Attention Branch"): angular-hash queries and keys, stably sort each by
 *     hash key, cut both sorted orders into blocks of b, and let query block t
 *     attend exactly to key block t, giving O_sparse and d_sparse;
 *   - the RACE low-rank branch (Section 3.1; Algorithm "RACE Low-Rank
 *     Attention Branch"): soft hypercube-hash features phi, bucket summaries
 *     A = Phi_K^T 1 and B = Phi_K^T V per table, and the table-averaged readout
 *     Num = Phi_Q B / L_s, Den = Phi_Q A / L_s, giving O_lr = Num / (Den + eps)
 *     and d_lr = Den;
 *   - the denominator-aware fusion (Eq. (5) and Eq. (6); Algorithm 1 steps
 *     6-8): m = d_sparse / (d_sparse + lambda d_lr + eps),
 *     O = g_sparse m O_sparse + g_lr O_lr.
 * The N x N score matrix is never formed.
 *
 * Conventions for every entry point:
 *   - All tensor pointers are DEVICE pointers owned by the caller; the
 *     library allocates no memory. Scratch space comes from the caller through
 *     the workspace argument, sized by elsaa_workspace_size().
 *   - Calls are asynchronous on the caller's CUDA stream (cudaStream_t passed
 *     as void*; NULL = the legacy default stream) and never synchronise.
 *     elsaa_forward also runs the RACE key side, which needs no sort, on a
 *     library-owned stream (one per host thread and device, created on first
 *     use, non-blocking), forked from the caller's stream after the call's
 *     first operation and joined back into it with events before the block
 *     kernel: the call's work stays ordered on the caller's stream as a unit
 *     and can be captured into a CUDA graph.
 *   - Arguments are validated on the host before any launch. The return value
 *     is ELSAA_OK or one of the ELSAA_ERR_* codes; elsaa_last_error() then
 *     holds a one-line description (thread-local).
 *   - Tensors are contiguous row-major. Q, K, V and O are [B, H, N, d_h] of
 *     the element type params.dtype; per-token arrays are [B, H, N].
 */
#ifndef ELSAA_H
#define ELSAA_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

#define ELSAA_ABI_VERSION 6

/* Return codes. */
#define ELSAA_OK 0
#define ELSAA_ERR_INVALID_ARG 1  /* null pointer, bad size, N % b != 0 ... */
#define ELSAA_ERR_UNSUPPORTED 2  /* valid per the paper, not built here    */
#define ELSAA_ERR_WORKSPACE 3    /* workspace null or smaller than needed  */
#define ELSAA_ERR_CUDA 4         /* a CUDA runtime call or launch failed   */
#define ELSAA_ERR_DEVICE 5       /* a kernel reported a fault in-band      */

/* Element type of Q, K, V and O. */
#define ELSAA_BF16 0
#define ELSAA_FP32 1

/* Kernel family selection (params.impl). */
#define ELSAA_IMPL_AUTO 0   /* tensor-core kernels where supported (bf16)   */
#define ELSAA_IMPL_SIMT 1   /* fp32 CUDA-core kernels for every step        */

typedef struct elsaa_params {
    int B, H, N, d_h;   /* Q, K, V are [B, H, N, d_h] (Section 3)            */
    int dtype;          /* ELSAA_BF16 or ELSAA_FP32                           */
    int causal;         /* 0: Algorithm 1 (non-causal); 1: Algorithm "Causal
                           ELSAA": the recursive causal sortLSH branch
                           (CausalSparse with SortLSH blocks and MergeLSE)
                           and the chunked causal RACE branch, fused with the
                           log-domain multiplier. Built for bf16, impl AUTO,
                           d_h 64 or 128, race_bits 4 with race_tables 4, 8
                           or 16, block_size 32/64/128/256, neighbor_blocks
                           0, and N = n_leaf 2^k where the recursion stops at
                           segments of n_leaf <= causal_base_len rows, a
                           multiple of 128 and of block_size (no odd-length
                           padding); ELSAA_ERR_UNSUPPORTED otherwise.        */
    int block_size;     /* b, keys per query (sortLSH block size; Table 7 "s").
                           Requires N % b == 0 and b % 32 == 0, b <= 1024.    */
    int sort_bits;      /* sortLSH hash bits n_s in [0, 8] (Table 7: 4-5);
                           0 gives the identity order                         */
    int gray_order;     /* 1: codes ordered by rank in the reflected Gray
                           sequence (adjacent buckets differ in one bit);
                           0: plain binary code order                         */
    int race_tables;    /* L_s >= 1                                           */
    int race_bits;      /* gamma in [1, 8]; R = 2^gamma buckets per table;
                           L_s * R <= 1024                                    */
    float beta;         /* RACE temperature beta >= 0                         */
    float eps;          /* numerical floor epsilon > 0 (Table 7: 1e-6)        */
    float scale;        /* score scale for sortLSH; 0 -> 1/sqrt(d_h)          */
    float lambda;       /* scalar lambda >= 0, used when lambda_tok is NULL   */
    int fusion_mode;    /* 0: ELSAA multiplier of Eq. (5);
                           1: Sort_Lsh_RACE ablation, m := 1 (Section 5)      */
    int impl;           /* ELSAA_IMPL_AUTO or ELSAA_IMPL_SIMT                 */
    int neighbor_blocks;/* r >= 0: query block t also attends to the r
                           neighbouring sorted key blocks on each side,
                           t - r .. t + r clipped to the N / b blocks
                           (Section 5's cost paragraph: (2r + 1) b keys per
                           query; the paper's runs use r = 0). bf16 with
                           b of 128 or 256, r = 1 and race_bits = 4 runs on
                           the tensor cores; other r > 0 shapes run the
                           sparse branch on CUDA cores (fp32).
                           elsaa_backward requires r = 0                  */
    int causal_chunk;   /* C >= 1, chunk length of causal RACE (Algorithm
                           "Causal RACE"). The result does not depend on C
                           (the prefix-state form is exact); the device
                           uses 128-token chunks. Ignored when causal = 0  */
    int causal_base_len;/* N_0 >= 1, segment length at which CausalSparse
                           switches to exact causal attention (Table 7,
                           "Sort_LSH min length"). Ignored when causal = 0 */
    int out_fp32;       /* 0: O has the element type dtype; 1: O is fp32
                           [B, H, N, d_h] whatever dtype is: the result is
                           not rounded to bf16 (the same arithmetic, with
                           the final rounding of a bf16 O left out). Not
                           used by elsaa_backward or elsaa_gates          */
    int selector;       /* keys of the sparse branch. 0: the sorted key
                           block (Algorithm sortLSH). 1: per-query top-k, a
                           selector Section 3 names as future work, read
                           here as: after the hash and stable sort, block
                           sums qbar_t, kbar_u of the sorted blocks (fp32,
                           sequential in sorted order); block scores
                           <qbar_t, kbar_u>; query block t takes key block
                           t and the topk_blocks - 1 other blocks of largest
                           score (ties: lower block); each query keeps the
                           topk candidate keys of largest <q_i, k_j> (ties:
                           lower key index) and runs the block step over
                           them. Every score is the sequential fp32 FMA
                           chain of the sort hash, so the selected sets
                           are exact. Requires causal = 0, neighbor_blocks
                           = 0, topk_blocks * block_size <= 512 and at most
                           8192 blocks per head; elsaa_backward returns
                           ELSAA_ERR_UNSUPPORTED                           */
    int topk;           /* selector 1: keys per query, 1 <= topk <=
                           topk_blocks * block_size                        */
    int topk_blocks;    /* selector 1: candidate key blocks per query
                           block, 1 <= topk_blocks <= N / block_size       */
} elsaa_params;

/*
 * Bytes of scratch memory elsaa_forward needs for these parameters.
 * Returns ELSAA_OK and writes *bytes, or ELSAA_ERR_INVALID_ARG /
 * ELSAA_ERR_UNSUPPORTED if the parameters would be rejected by
 * elsaa_forward. No CUDA call is made.
 */
int elsaa_workspace_size(const elsaa_params *params, size_t *bytes);

/*
 * ELSAA forward pass for all B*H heads (Algorithm 1 steps 4-8, without the
 * Q/K/V and output projections, which stay dense outside the operator).
 *
 * q, k, v      [B, H, N, d_h] of params->dtype (device, read only). q, k, v,
 *              o and w_race must be 16-byte aligned (rows move in 16-byte
 *              pieces); ELSAA_ERR_INVALID_ARG otherwise.
 * w_sort       [H, sort_bits, d_h] fp32: planes of the angular sort hash,
 *              shared by queries and keys of head h; may be NULL when
 *              sort_bits == 0. Bit p of x is [<w_sort[h][p], x> > 0], the
 *              projection evaluated as a sequential fp32 fused multiply-add
 *              chain over i = 0..d_h-1.
 * w_race       [H, L_s, gamma, d_h] fp32: Gaussian rows W^(l) of Algorithm
 *              RACE. The tensor-core path rounds them to bf16; pass
 *              bf16-representable values for bit-comparable results.
 * lambda_tok   [B, H, N] fp32 per-token lambda_i >= 0, or NULL for the scalar
 *              params->lambda (Section 3.3: fixed, learned scalar or
 *              query-dependent).
 * gates        [B, H, N, 2] fp32 (g_sparse, g_lr) per token, or NULL for
 *              (1, 1). The paper's gates are sigma(G_theta(q_i)); the gate
 *              network itself runs outside the operator.
 * o            [B, H, N, d_h] of params->dtype, or fp32 with
 *              params->out_fp32 = 1 (device, written).
 * log_d_sparse [B, H, N] fp32 log of the sparse denominator, or NULL.
 * d_lr         [B, H, N] fp32 low-rank denominator Den, or NULL.
 * m_sparse     [B, H, N] fp32 multiplier of Eq. (5), or NULL.
 * perm_q/k     [B, H, N] int32 sorted orders P_Q, P_K (sorted position ->
 *              original index; equal keys by increasing index), or NULL.
 * workspace    device scratch of at least elsaa_workspace_size() bytes,
 *              256-byte aligned. Its contents need no initialisation.
 * stream       cudaStream_t (as void*) on which all work is enqueued.
 *
 * With params->causal = 1 the same call runs Algorithm "Causal ELSAA":
 * o, log_d_sparse (log of the merged CausalSparse denominator), d_lr (the
 * causal Den) and m_sparse keep their meanings; perm_q and perm_k are not
 * written (each level of the recursion sorts its own halves: see
 * elsaa_causal_index_lists).
 *
 * Errors: ELSAA_ERR_INVALID_ARG / _UNSUPPORTED / _WORKSPACE before any
 * launch; ELSAA_ERR_CUDA if a launch fails (the message names the kernel).
 */
int elsaa_forward(const elsaa_params *params, const void *q, const void *k,
                  const void *v, const float *w_sort, const float *w_race,
                  const float *lambda_tok, const float *gates, void *o,
                  float *log_d_sparse, float *d_lr, float *m_sparse,
                  int32_t *perm_q, int32_t *perm_k, void *workspace,
                  size_t workspace_bytes, void *stream);

/*
 * elsaa_forward for callers that cannot allocate device memory.
 *
 * Not part of the paper's method (the paper has no counterpart); it exists
 * for deployment. Some callers have no way to obtain scratch memory: a
 * plug-in whose host application owns every device buffer and offers no
 * allocator, or code on a latency-critical path that must not call
 * cudaMalloc / cudaFree because those calls can synchronise the whole
 * device. Such callers still own and pass the inputs and outputs exactly as
 * for elsaa_forward (same meaning, layout and errors), but no workspace.
 *
 * Scratch comes from one fixed array of ELSAA_STATIC_WORKSPACE_BYTES inside
 * the library's device image. Every GPU on which the library's kernels are
 * loaded reserves that memory until the process exits.
 *  - Every call looks up the array's device address on the current device
 *    (cudaGetSymbolAddress: a query, not an allocation), so a device reset
 *    leaves no stale address behind. The first call on a device may load
 *    the library's module there; make it before any stream capture.
 *  - Problems whose elsaa_workspace_size() exceeds the array are rejected
 *    with ELSAA_ERR_WORKSPACE (the message gives both sizes); nothing is
 *    launched.
 *  - All calls share the one array and it keeps the previous call's
 *    contents. The forward pass writes every scratch value before reading
 *    it (the status word is cleared at the start of each call). Calls whose
 *    GPU work overlaps (other streams, other host threads without ordering)
 *    race on the array and produce wrong results: order them on one stream.
 *  - Allocates nothing: no cudaMalloc, cudaFree or allocating library call.
 */
#define ELSAA_STATIC_WORKSPACE_BYTES ((size_t)64 << 20)

int elsaa_forward_noalloc(const elsaa_params *params, const void *q,
                          const void *k, const void *v, const float *w_sort,
                          const float *w_race, const float *lambda_tok,
                          const float *gates, void *o, float *log_d_sparse,
                          float *d_lr, float *m_sparse, int32_t *perm_q,
                          int32_t *perm_k, void *stream);

/*
 * elsaa_check_status for elsaa_forward_noalloc, whose callers never see the
 * static array's address: synchronises `stream` and reads the status word
 * that the last elsaa_forward_noalloc wrote at the start of the array
 * (bounded waits that ran out, inconsistent sort counts). Returns as
 * elsaa_check_status. Read it before the next call overwrites the word.
 */
int elsaa_check_status_noalloc(void *stream);

/*
 * elsaa_selftest_wait_timeout on the static array (see that function): lets
 * a test see elsaa_check_status_noalloc report a timed-out wait without any
 * fault. The next elsaa_forward_noalloc clears the word.
 */
int elsaa_selftest_wait_timeout_noalloc(int limit_ms, void *stream);

/*
 * Backward pass: gradients of a loss L with respect to Q, K, V (and
 * optionally the gates and the per-token lambda), given dO = dL/dO.
 *
 * The paper trains ELSAA end to end but prints no backward pass; this is
 * the derivative of the forward definitions (Algorithm "sortLSH Sparse
 * Exact Attention Branch" block step, Algorithm "RACE Low-Rank Attention
 * Branch", Eq. (5)-(6)). The hash and the sort are piecewise constant and
 * carry no gradient: the caller passes the permutations perm_q, perm_k that
 * elsaa_forward returned for the same inputs (required, not recomputed).
 * The RACE summaries A and B are taken from race_A, race_B when given
 * (saved from the forward with elsaa_forward_race_summaries) and
 * recomputed otherwise; block scores and features are always recomputed.
 *
 * params, q, k, v, w_sort, w_race, lambda_tok, gates: as for elsaa_forward
 *              (w_sort is not read).
 * d_o          [B, H, N, d_h] of params->dtype: dL/dO (device, read only).
 * perm_q/k     [B, H, N] int32 from elsaa_forward (device, read only).
 * dq, dk, dv   [B, H, N, d_h] fp32 (device, written).
 * d_gates      [B, H, N, 2] fp32 dL/d(g_sparse, g_lr), or NULL.
 * d_lambda     [B, H, N] fp32 dL/dlambda_i, or NULL.
 * race_A       [B, H, r] fp32 and race_B [B, H, r, d_h] fp32: the forward's
 *              summaries (device, read only), both or neither (NULL, NULL:
 *              recomputed); 16-byte aligned.
 * workspace    at least elsaa_backward_workspace_size() bytes, 256-byte
 *              aligned (a different size from the forward workspace).
 *
 * Paths: with impl AUTO, bf16, b = 64, d_h = 64, race_bits 4 with
 * race_tables 4 or 8 and N a multiple of 128, the products run on the
 * tensor cores (bf16 operands, fp32 accumulation; gradients within about
 * 1e-2 of the largest gradient magnitude); otherwise on CUDA cores in fp32
 * (all dtypes) for the forward's shapes with b * (4 d_h + b + r + 2) * 4
 * bytes of block state <= 200 KiB (e.g. b = 64, d_h = 64, r = 128);
 * ELSAA_ERR_UNSUPPORTED otherwise and for causal = 1. Errors as for
 * elsaa_forward.
 */
int elsaa_backward_workspace_size(const elsaa_params *params, size_t *bytes);
int elsaa_backward(const elsaa_params *params, const void *q, const void *k,
                   const void *v, const float *w_sort, const float *w_race,
                   const float *lambda_tok, const float *gates,
                   const void *d_o, const int32_t *perm_q,
                   const int32_t *perm_k, float *dq, float *dk, float *dv,
                   float *d_gates, float *d_lambda, const float *race_A,
                   const float *race_B, void *workspace,
                   size_t workspace_bytes, void *stream);

/*
 * Copies the RACE summaries of the last elsaa_forward enqueued with this
 * `params` and `workspace` (Algorithm "RACE Low-Rank Attention Branch",
 * steps 5-7: A = Phi_K^T 1, B = Phi_K^T V, per table and bucket, summed over
 * all keys) into race_A [B, H, r] and race_B [B, H, r, d_h] (fp32, device,
 * written), stream-ordered after that forward on `stream`: the saved
 * activations elsaa_backward can take instead of recomputing them.
 * ELSAA_ERR_UNSUPPORTED for causal = 1 (its RACE branch keeps per-chunk
 * prefix states instead); other errors as for elsaa_forward.
 */
int elsaa_forward_race_summaries(const elsaa_params *params,
                                 const void *workspace,
                                 size_t workspace_bytes, float *race_A,
                                 float *race_B, void *stream);

/*
 * The selection of the causal sparse branch (Algorithm "Causal sortLSH
 * Sparse Exact Attention Branch"): every node of the recursion above the
 * base segments calls SortLSH on its future half's queries and its past
 * half's keys, each stably sorted by sort code; sorted query block t of the
 * node attends exactly to sorted key block t.
 *
 * elsaa_causal_levels writes the number Lv of halving levels for params
 * (N = n_leaf 2^Lv, n_leaf <= causal_base_len; 0 when N fits one segment).
 *
 * elsaa_causal_index_lists copies the sorted orders of the last causal
 * elsaa_forward enqueued with this `params` and `workspace` into `lists`
 * (device, written, stream-ordered after that forward on `stream`):
 *     lists[l - 1][w][b][h][j m + p],  l = 1..Lv (1 = the top level),
 *     m = N / 2^l rows per half, node j in [0, 2^(l-1)), p in [0, m),
 * w = 0: the token index (within the head) of the future-half query at
 * sorted position p of node j, whose half is rows [(2j+1) m, (2j+2) m);
 * w = 1: the same for the past-half keys, rows [2j m, (2j+1) m). Equal codes
 * keep increasing token order. Query at sorted position p attends to the
 * keys at sorted positions [floor(p / b) b, floor(p / b) b + b) of the same
 * node. Lv * 2 * B * H * N / 2 int32 values; nothing is copied when Lv = 0.
 * Errors as for elsaa_forward_race_summaries; ELSAA_ERR_INVALID_ARG unless
 * params->causal = 1.
 */
int elsaa_causal_levels(const elsaa_params *params, int *levels);
int elsaa_causal_index_lists(const elsaa_params *params,
                             const void *workspace, size_t workspace_bytes,
                             int32_t *lists, void *stream);

/*
 * The key sets of the last elsaa_forward with params->selector = 1 enqueued
 * with this `params` and `workspace`: keys[b][h][i][0 .. topk) = the
 * original indices of the keys query i attends, increasing (device, int32,
 * written, stream-ordered after that forward on `stream`).
 * ELSAA_ERR_INVALID_ARG unless params->selector = 1; other errors as for
 * elsaa_forward_race_summaries.
 */
int elsaa_forward_selected_keys(const elsaa_params *params,
                                const void *workspace, size_t workspace_bytes,
                                int32_t *keys, void *stream);

/*
 * Token-wise gates and query-dependent lambda, the learned inputs of the
 * fusion (Section 3.3: (g_sparse,i, g_lr,i) = sigma(G_theta(q_i)); the
 * experiment-hyperparameter appendix (Appendix D): G_theta is a two-layer
 * MLP with a SiLU hidden layer and two independent sigmoid outputs, and the
 * input-dependent coefficient lambda_i = c + sigma(w^T q_i + b), floored at
 * lambda_min). For every query row q_i of head h:
 *     a_i         = SiLU(W1[h] q_i + b1[h])            (width g)
 *     gates[i]    = sigmoid(W2[h] a_i + b2[h])         (2 values)
 *     lambda_tok[i] = max(c[h] + sigmoid(w_lambda[h] . q_i + b_lambda[h]),
 *                         lambda_min)
 * with SiLU(x) = x sigmoid(x). The outputs have exactly the layouts of
 * elsaa_forward's `gates` and `lambda_tok` arguments: enqueue elsaa_gates
 * and then elsaa_forward on one stream for the full fusion with learned
 * gates. Parameter gradients of the MLP are not computed (elsaa_backward
 * returns dL/dgates and dL/dlambda, from which they follow).
 */
typedef struct elsaa_gate_mlp {
    int hidden;              /* g, a multiple of 16 in [16, 128]
                                (the paper uses 64 or 128)                  */
    const float *w1;         /* [H, g, d_h]; the tensor-core path rounds it
                                to bf16: pass bf16-representable values     */
    const float *b1;         /* [H, g]                                      */
    const float *w2;         /* [H, 2, g]: rows for g_sparse, g_lr          */
    const float *b2;         /* [H, 2]                                      */
    const float *w_lambda;   /* [H, d_h] (bf16-representable), or NULL for
                                no lambda output                            */
    const float *b_lambda;   /* [H]; required with w_lambda                 */
    const float *c_lambda;   /* [H], >= 0; required with w_lambda           */
    float lambda_min;        /* > 0 (the paper: 1e-6)                       */
} elsaa_gate_mlp;

/*
 * q           [B, H, N, d_h] of params->dtype (device, 16-byte aligned).
 * gates       [B, H, N, 2] fp32 (device, written, 8-byte aligned).
 * lambda_tok  [B, H, N] fp32 (device, written); required when
 *             mlp->w_lambda != NULL, ignored otherwise.
 * workspace   at least elsaa_gates_workspace_size() bytes, 256-byte
 *             aligned (holds the bf16 image of W1 and w_lambda and the
 *             status word that elsaa_check_status reads).
 * All parameter arrays are device pointers; b1 and w2 must be 16-byte
 * aligned (rows are read in 16-byte pieces). params is validated as for
 * elsaa_forward. bf16 inputs with d_h in {64, 128} run on the tensor cores
 * (tcgen05, fp32 accumulation); other shapes and fp32 inputs on CUDA cores
 * in fp32. Errors: ELSAA_ERR_INVALID_ARG / _UNSUPPORTED / _WORKSPACE before
 * any launch, ELSAA_ERR_CUDA if a launch fails.
 */
int elsaa_gates_workspace_size(const elsaa_params *params,
                               const elsaa_gate_mlp *mlp, size_t *bytes);
int elsaa_gates(const elsaa_params *params, const elsaa_gate_mlp *mlp,
                const void *q, float *gates, float *lambda_tok,
                void *workspace, size_t workspace_bytes, void *stream);

/*
 * The forward pass with its learned gates and query-dependent lambda
 * computed in the same call: the result of elsaa_gates followed by
 * elsaa_forward with those gates and lambda_tok (Section 3.3 fusion with
 * gates sigma(G_theta(q_i)); Appendix D's gate MLP and input-dependent
 * lambda_i).
 *
 * Non-causal: the gate kernel runs on the caller's stream right after the
 * sort, while the RACE key side (the longer of the two chains before the
 * block kernel) is still running, so it fills the SMs the sort chain has
 * left idle; the block kernel then reads the gates and lambda. Causal: the
 * gate kernel, then the causal forward.
 *
 * Arguments as elsaa_forward and elsaa_gates; gates_out [B, H, N, 2] and
 * lambda_out [B, H, N] (fp32, device, written) are optional copies of the
 * computed gates and lambda (NULL: kept in the workspace; lambda is only
 * computed when mlp->w_lambda is given, otherwise params->lambda is used).
 * workspace: at least elsaa_forward_gated_workspace_size() bytes, 256-byte
 * aligned. Errors as for elsaa_forward and elsaa_gates.
 */
int elsaa_forward_gated_workspace_size(const elsaa_params *params,
                                       const elsaa_gate_mlp *mlp,
                                       size_t *bytes);
int elsaa_forward_gated(const elsaa_params *params,
                        const elsaa_gate_mlp *mlp, const void *q,
                        const void *k, const void *v, const float *w_sort,
                        const float *w_race, void *o, float *log_d_sparse,
                        float *d_lr, float *m_sparse, int32_t *perm_q,
                        int32_t *perm_k, float *gates_out, float *lambda_out,
                        void *workspace, size_t workspace_bytes,
                        void *stream);

/*
 * Synchronises `stream` and reads the in-band status word that the kernels
 * of the last elsaa_forward on this workspace wrote (bounded waits that ran
 * out, inconsistent sort counts). Returns ELSAA_OK, ELSAA_ERR_DEVICE (with
 * the recorded code in elsaa_last_error()) or ELSAA_ERR_CUDA.
 */
int elsaa_check_status(const void *workspace, void *stream);

/*
 * Per-kernel timing for measurement tools. Between elsaa_profile_start() and
 * elsaa_profile_stop(), every kernel elsaa_forward launches is bracketed by
 * a pair of CUDA events recorded on the caller's stream. elsaa_profile_stop
 * waits for those events and writes one entry per kernel name (launch count,
 * summed device milliseconds) into out[0..max_entries), setting *n_entries.
 * Not for use during CUDA graph capture. Returns ELSAA_OK or ELSAA_ERR_CUDA.
 */
typedef struct elsaa_kernel_stat {
    char name[32];
    int launches;
    double total_ms;
} elsaa_kernel_stat;

int elsaa_profile_start(void);
int elsaa_profile_stop(elsaa_kernel_stat *out, int max_entries,
                       int *n_entries);

/*
 * Self-test of the in-band failure path, for tests. Every wait inside the
 * kernels is bounded; one that runs out records {code 3 (wait timeout),
 * site, CTA} in the workspace status word and lets its kernel return, and
 * elsaa_check_status reports it. This call enqueues one CTA whose bounded
 * mbarrier wait can never complete (nothing arrives): after limit_ms
 * milliseconds (1..2000) it records the timeout at site 0x7e57 and returns.
 * Nothing faults or hangs; the context stays usable and the next
 * elsaa_forward on the workspace clears the word. workspace: 256-byte
 * aligned, at least 16 bytes.
 */
int elsaa_selftest_wait_timeout(void *workspace, size_t workspace_bytes,
                                int limit_ms, void *stream);

/* One-line description of the last error on this thread ("" if none). */
const char *elsaa_last_error(void);

/* ELSAA_ABI_VERSION of the loaded library. */
int elsaa_abi_version(void);

#ifdef __cplusplus
}
#endif

#endif /* ELSAA_H */
