// C ABI of libelsaa: argument validation, workspace plan, launch sequence.
#include <math.h>
#include <stdarg.h>
#include <stdio.h>
#include <string.h>

#include <cudaTypedefs.h>

#include <deque>
#include <mutex>
#include <string>
#include <vector>

#include "internal.h"

namespace elsaa {

namespace {

thread_local char g_err[512] = "";

int fail(int code, const char *fmt, ...) {
    va_list ap;
    va_start(ap, fmt);
    vsnprintf(g_err, sizeof(g_err), fmt, ap);
    va_end(ap);
    return code;
}

size_t align_up(size_t x, size_t a) { return (x + a - 1) / a * a; }

// Optional per-launch event timing (elsaa_profile_start / _stop).
struct ProfRec {
    const char *name;
    cudaEvent_t a, b;
};
std::mutex g_prof_mu;
bool g_prof_on = false;
std::vector<ProfRec> g_prof;
std::vector<cudaEvent_t> g_ev_pool;

cudaEvent_t pool_event() {
    if (!g_ev_pool.empty()) {
        cudaEvent_t e = g_ev_pool.back();
        g_ev_pool.pop_back();
        return e;
    }
    cudaEvent_t e = nullptr;
    cudaEventCreate(&e);
    return e;
}

// Launches `fn` on `st`, bracketed by events when profiling is on.
template <typename F>
cudaError_t timed(const char *name, cudaStream_t st, F fn) {
    if (!g_prof_on) return fn();
    std::lock_guard<std::mutex> lk(g_prof_mu);
    ProfRec r{name, pool_event(), pool_event()};
    cudaEventRecord(r.a, st);
    cudaError_t e = fn();
    cudaEventRecord(r.b, st);
    g_prof.push_back(r);
    return e;
}

// A second stream per host thread and device for the RACE key side, which
// needs no sort: forked from the caller's stream after the status reset and
// joined back before the block kernel, so it overlaps the hash, scan and
// scatter. Created on first use, kept for the life of the process.
struct SideStream {
    int dev = -1;
    cudaStream_t s = nullptr;
    cudaEvent_t fork = nullptr, join = nullptr;
};

cudaError_t side_stream(SideStream **out) {
    // a deque keeps earlier entries in place when another device is added
    thread_local std::deque<SideStream> ss;
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    for (auto &x : ss)
        if (x.dev == dev) {
            *out = &x;
            return cudaSuccess;
        }
    SideStream x;
    x.dev = dev;
    e = cudaStreamCreateWithFlags(&x.s, cudaStreamNonBlocking);
    if (e == cudaSuccess)
        e = cudaEventCreateWithFlags(&x.fork, cudaEventDisableTiming);
    if (e == cudaSuccess)
        e = cudaEventCreateWithFlags(&x.join, cudaEventDisableTiming);
    if (e != cudaSuccess) return e;
    ss.push_back(x);
    *out = &ss.back();
    return cudaSuccess;
}

// RACE key-chunk CTAs aimed for: about two per SM of a 152-SM GB300. A
// constant (not a device query) keeps the workspace size device-independent.
constexpr long kRaceTargetCtas = 304;

}  // namespace

int make_plan(const elsaa_params *p, Plan *P, const char **msg) {
    auto bad = [&](int code, const char *m) {
        *msg = m;
        return code;
    };
    if (!p) return bad(ELSAA_ERR_INVALID_ARG, "params is NULL");
    if (p->B <= 0 || p->H <= 0 || p->N <= 0 || p->d_h <= 0)
        return bad(ELSAA_ERR_INVALID_ARG, "B, H, N and d_h must be positive");
    if (p->dtype != ELSAA_BF16 && p->dtype != ELSAA_FP32)
        return bad(ELSAA_ERR_INVALID_ARG, "dtype must be ELSAA_BF16 or ELSAA_FP32");
    if (p->causal != 0 && p->causal != 1)
        return bad(ELSAA_ERR_INVALID_ARG, "causal must be 0 or 1");
    if (p->block_size <= 0)
        return bad(ELSAA_ERR_INVALID_ARG, "block_size must be positive");
    if (p->N % p->block_size != 0)
        return bad(ELSAA_ERR_INVALID_ARG, "N must be a multiple of block_size");
    if (p->block_size % 32 != 0 || p->block_size > 1024)
        return bad(ELSAA_ERR_UNSUPPORTED,
                   "block_size must be a multiple of 32 and at most 1024");
    if (p->d_h != 32 && p->d_h != 64 && p->d_h != 128)
        return bad(ELSAA_ERR_UNSUPPORTED, "d_h must be 32, 64 or 128");
    if (p->sort_bits < 0 || p->sort_bits > 16)
        return bad(ELSAA_ERR_INVALID_ARG, "sort_bits must be in [0, 16]");
    if (p->sort_bits > 8)
        return bad(ELSAA_ERR_UNSUPPORTED, "sort_bits above 8 are not built");
    if (p->gray_order != 0 && p->gray_order != 1)
        return bad(ELSAA_ERR_INVALID_ARG, "gray_order must be 0 or 1");
    if (p->race_tables < 1 || p->race_bits < 1 || p->race_bits > 8)
        return bad(ELSAA_ERR_INVALID_ARG,
                   "race_tables must be >= 1 and race_bits in [1, 8]");
    if ((long)p->race_tables << p->race_bits > 1024)
        return bad(ELSAA_ERR_UNSUPPORTED, "race_tables * 2^race_bits > 1024");
    if (!(p->beta >= 0.f) || !isfinite(p->beta))
        return bad(ELSAA_ERR_INVALID_ARG, "beta must be finite and >= 0");
    if (!(p->eps > 0.f) || !isfinite(p->eps))
        return bad(ELSAA_ERR_INVALID_ARG, "eps must be finite and > 0");
    if (!(p->scale >= 0.f) || !isfinite(p->scale))
        return bad(ELSAA_ERR_INVALID_ARG, "scale must be finite and >= 0");
    if (!(p->lambda >= 0.f) || !isfinite(p->lambda))
        return bad(ELSAA_ERR_INVALID_ARG, "lambda must be finite and >= 0");
    if (p->fusion_mode != 0 && p->fusion_mode != 1)
        return bad(ELSAA_ERR_INVALID_ARG, "fusion_mode must be 0 or 1");
    if (p->impl != ELSAA_IMPL_AUTO && p->impl != ELSAA_IMPL_SIMT)
        return bad(ELSAA_ERR_INVALID_ARG, "impl must be AUTO or SIMT");
    if (p->neighbor_blocks < 0)
        return bad(ELSAA_ERR_INVALID_ARG, "neighbor_blocks must be >= 0");
    if (p->out_fp32 != 0 && p->out_fp32 != 1)
        return bad(ELSAA_ERR_INVALID_ARG, "out_fp32 must be 0 or 1");
    if (p->selector != 0 && p->selector != 1)
        return bad(ELSAA_ERR_INVALID_ARG, "selector must be 0 or 1");
    if (p->selector == 1) {
        if (p->topk_blocks < 1 || p->topk_blocks > p->N / p->block_size)
            return bad(ELSAA_ERR_INVALID_ARG,
                       "selector 1: topk_blocks must be in [1, N / block_size]");
        if (p->topk < 1 || (long)p->topk > (long)p->topk_blocks * p->block_size)
            return bad(ELSAA_ERR_INVALID_ARG,
                       "selector 1: topk must be in [1, topk_blocks * "
                       "block_size]");
        if (p->neighbor_blocks != 0)
            return bad(ELSAA_ERR_INVALID_ARG,
                       "selector 1: neighbor_blocks must be 0 (the candidate "
                       "blocks replace the neighbour window)");
        if (p->causal != 0)
            return bad(ELSAA_ERR_UNSUPPORTED,
                       "selector 1 is not built for the causal variant");
    }
    if ((long)p->B * p->H > 65535)
        return bad(ELSAA_ERR_UNSUPPORTED, "B * H must be at most 65535");
    if ((long)p->B * p->H * p->N > (1L << 31) - 1)
        return bad(ELSAA_ERR_UNSUPPORTED, "B * H * N must fit in int32");

    Plan &Q = *P;
    Q = Plan{};
    Q.B = p->B;
    Q.H = p->H;
    Q.N = p->N;
    Q.d = p->d_h;
    Q.BH = p->B * p->H;
    Q.dtype = p->dtype;
    Q.b = p->block_size;
    Q.n_s = p->sort_bits;
    Q.bins = 1 << p->sort_bits;
    Q.gray = p->gray_order;
    Q.L = p->race_tables;
    Q.gamma = p->race_bits;
    Q.R = 1 << p->race_bits;
    Q.r = Q.L * Q.R;
    Q.tables_per_slice = Q.R >= kSliceBuckets ? 1 : kSliceBuckets / Q.R;
    if (Q.R > kSliceBuckets)
        return bad(ELSAA_ERR_UNSUPPORTED, "race_bits above 6 are not built");
    Q.slices = (Q.L + Q.tables_per_slice - 1) / Q.tables_per_slice;
    Q.beta = p->beta;
    Q.eps = p->eps;
    Q.scale = p->scale > 0.f ? p->scale : 1.0f / sqrtf((float)p->d_h);
    Q.lambda = p->lambda;
    Q.fusion_mode = p->fusion_mode;
    Q.o32 = p->dtype == ELSAA_BF16 && p->out_fp32 == 1;
    Q.sel = p->selector;
    Q.tk_k = Q.sel ? p->topk : 0;
    Q.tk_c = Q.sel ? p->topk_blocks : 0;
    // neighbour windows wider than the sequence change nothing: clip
    Q.nb = p->neighbor_blocks < Q.N / Q.b ? p->neighbor_blocks : Q.N / Q.b;
    Q.impl = 1;
    Q.Lg_pad = (Q.L * Q.gamma + 15) / 16 * 16;
    Q.tiles = (Q.N + kHashTile - 1) / kHashTile;
    if (p->impl == ELSAA_IMPL_AUTO && tc_supported(Q)) {
        // tensor-core path: one wave of 128-key-tile chunks per head
        Q.impl = 2;
        Q.S = tc_race_chunks(Q, &Q.chunk);
    } else {
        // RACE key chunks: enough CTAs for about two waves, 32-key steps.
        long want = (kRaceTargetCtas + (long)Q.BH * Q.slices - 1) /
                    ((long)Q.BH * Q.slices);
        long maxS = (Q.N + 31) / 32;
        long S = want < 1 ? 1 : (want > maxS ? maxS : want);
        long chunk = ((Q.N + S - 1) / S + 31) / 32 * 32;
        Q.chunk = (int)chunk;
        Q.S = (int)((Q.N + chunk - 1) / chunk);
    }
    size_t BHN = (size_t)Q.BH * Q.N;
    size_t off = 0;
    Q.off_status = off;
    off = align_up(off + sizeof(DeviceStatus), 256);
    Q.off_keyrank = off;
    off = align_up(off + 2 * BHN * sizeof(uint32_t), 256);
    Q.off_hist = off;
    off = align_up(off + (size_t)2 * Q.BH * Q.tiles * Q.bins * sizeof(int), 256);
    Q.off_perm = off;
    off = align_up(off + 2 * BHN * sizeof(int32_t), 256);
    Q.off_part = off;
    off = align_up(off + (size_t)Q.BH * Q.S * ((size_t)Q.r * Q.d + Q.r) *
                             sizeof(float), 256);
    Q.off_A = off;
    off = align_up(off + (size_t)Q.BH * Q.r * sizeof(float), 256);
    Q.off_B = off;
    off = align_up(off + (size_t)Q.BH * Q.r * Q.d * sizeof(float), 256);
    Q.off_Bh = off;
    off = align_up(off + (size_t)Q.BH * Q.r * Q.d * sizeof(uint16_t), 256);
    Q.off_W = off;
    off = align_up(off + (size_t)Q.H * Q.Lg_pad * Q.d * sizeof(uint16_t), 256);
    Q.off_sums = Q.off_cand = Q.off_mask = off;
    if (Q.sel) {
        if (!topk_supported(Q, msg)) return ELSAA_ERR_UNSUPPORTED;
        const size_t T = (size_t)(Q.N / Q.b);
        Q.off_sums = off;  // [2][BH][T][d] fp32 block sums
        off = align_up(off + 2 * Q.BH * T * Q.d * sizeof(float), 256);
        Q.off_cand = off;  // [BH][T][c] candidate blocks
        off = align_up(off + Q.BH * T * Q.tk_c * sizeof(int32_t), 256);
        Q.off_mask = off;  // [BH][N][c b / 32] selected candidates
        off = align_up(off + BHN * (Q.tk_c * Q.b / 32) * sizeof(uint32_t),
                       256);
    }
    Q.total = off;
    *msg = "";
    return ELSAA_OK;
}

namespace {

cudaError_t encode_2d(CUtensorMap *map, CUtensorMapDataType type,
                      uint32_t esize, const void *base, uint64_t rows,
                      uint64_t cols, uint32_t box_cols, uint32_t box_rows,
                      CUtensorMapSwizzle swizzle) {
    static PFN_cuTensorMapEncodeTiled_v12000 encode = nullptr;
    static std::once_flag once;
    std::call_once(once, [] {
        void *fn = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPoint("cuTensorMapEncodeTiled", &fn,
                                    cudaEnableDefault, &q) == cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            encode = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(fn);
    });
    if (!encode) return cudaErrorNotSupported;
    cuuint64_t dims[2] = {cols, rows};
    cuuint64_t strides[1] = {cols * esize};
    cuuint32_t box[2] = {box_cols, box_rows};
    cuuint32_t estr[2] = {1, 1};
    CUresult r = encode(map, type, 2,
                        const_cast<void *>(base), dims, strides, box, estr,
                        CU_TENSOR_MAP_INTERLEAVE_NONE, swizzle,
                        CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                        CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    return r == CUDA_SUCCESS ? cudaSuccess : cudaErrorInvalidValue;
}

}  // namespace

cudaError_t make_tma_map_bf16(CUtensorMap *map, const void *base,
                              uint64_t rows, uint64_t cols,
                              uint32_t box_rows) {
    return encode_2d(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, base, rows,
                     cols, 64, box_rows, CU_TENSOR_MAP_SWIZZLE_128B);
}

cudaError_t make_tma_map_f32(CUtensorMap *map, const void *base,
                             uint64_t rows, uint64_t cols, uint32_t box_cols,
                             uint32_t box_rows) {
    if (box_cols != 32) return cudaErrorInvalidValue;
    return encode_2d(map, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 4, base, rows,
                     cols, box_cols, box_rows, CU_TENSOR_MAP_SWIZZLE_128B);
}

cudaError_t make_tma_map_bf16_narrow(CUtensorMap *map, const void *base,
                                     uint64_t rows, uint64_t cols,
                                     uint32_t box_cols, uint32_t box_rows) {
    CUtensorMapSwizzle sw;
    switch (box_cols) {
        case 16: sw = CU_TENSOR_MAP_SWIZZLE_32B; break;
        case 32: sw = CU_TENSOR_MAP_SWIZZLE_64B; break;
        case 64: sw = CU_TENSOR_MAP_SWIZZLE_128B; break;
        default: return cudaErrorInvalidValue;
    }
    return encode_2d(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, base, rows,
                     cols, box_cols, box_rows, sw);
}

int set_last_error(int code, const char *fmt, ...) {
    va_list ap;
    va_start(ap, fmt);
    vsnprintf(g_err, sizeof(g_err), fmt, ap);
    va_end(ap);
    return code;
}

}  // namespace elsaa

using namespace elsaa;

#define ELSAA_CHECK_LAUNCH(expr, name)                                       \
    do {                                                                     \
        cudaError_t e_ = (expr);                                             \
        if (e_ != cudaSuccess)                                               \
            return fail(ELSAA_ERR_CUDA, "%s: %s", name,                      \
                        cudaGetErrorString(e_));                             \
    } while (0)

namespace {

// Causal forward (Algorithm "Causal ELSAA"). Workspace: status | codes
// (sort hash, [2][B*H][N]) | tile histograms of the hash | per level and
// side the sorted halves [Lv][2][B*H][N / 2] | running sparse result O
// [B*H][N][d_h] fp32 and log d [B*H][N] | RACE segment summaries, then
// offsets [B*H][segments][r d_h + r] | prefix states sB (bf16) and sA of
// every 128-key chunk | bf16 planes | work counters.
struct CausalPlan {
    Plan P;   // geometry and the forward's hash / RACE settings
    Plan Pc;  // P with RACE chunks of 128 keys
    int Lv, n_leaf;
    size_t off_status, off_keyrank, off_hist, off_perms, off_RO, off_RL,
        off_part, off_sB, off_sA, off_W, off_ctr, total;
};

int make_causal_plan(const elsaa_params *p, CausalPlan *C, const char **msg) {
    if (p->causal_chunk < 1 || p->causal_base_len < 1) {
        *msg = "causal_chunk and causal_base_len must be >= 1";
        return ELSAA_ERR_INVALID_ARG;
    }
    int rc = make_plan(p, &C->P, msg);
    if (rc != ELSAA_OK) return rc;
    const Plan &P = C->P;
    if (P.nb != 0) {
        *msg = "the causal variant requires neighbor_blocks = 0";
        return ELSAA_ERR_UNSUPPORTED;
    }
    // unrolled recursion: halve until a segment fits the base length
    int n = P.N, Lv = 0;
    while (n > p->causal_base_len) {
        if (n % 2) {
            *msg = "causal: this N and causal_base_len make the recursion pad "
                   "an odd-length segment (built: N = n_leaf 2^k with "
                   "n_leaf <= causal_base_len)";
            return ELSAA_ERR_UNSUPPORTED;
        }
        n /= 2;
        ++Lv;
    }
    C->Lv = Lv;
    C->n_leaf = n;
    if (!causal_tc_supported(P, n)) {
        *msg = "causal: built for bf16 with impl AUTO, d_h of 64 or 128, "
               "race_bits 4 with race_tables 4, 8 or 16, block_size 32, 64, "
               "128 or 256 dividing the base segments, base segments a "
               "multiple of 128 rows";
        return ELSAA_ERR_UNSUPPORTED;
    }
    // RACE key summaries of segments of whole 128-key chunks
    const int nseg = causal_segments(P);
    C->Pc = P;
    C->Pc.S = nseg;
    C->Pc.chunk = P.N / nseg;
    const size_t BHN = (size_t)P.BH * P.N;
    const size_t nc = (size_t)P.N / 128;
    size_t off = 0;
    C->off_status = off;
    off = align_up(off + sizeof(DeviceStatus), 256);
    C->off_keyrank = off;
    off = align_up(off + 2 * BHN * sizeof(uint32_t), 256);
    C->off_hist = off;
    off = align_up(off + (size_t)2 * P.BH * P.tiles * P.bins * sizeof(int),
                   256);
    C->off_perms = off;
    off = align_up(off + (size_t)Lv * BHN * sizeof(int32_t), 256);
    C->off_RO = off;
    off = align_up(off + BHN * P.d * sizeof(float), 256);
    C->off_RL = off;
    off = align_up(off + BHN * sizeof(float), 256);
    C->off_part = off;
    off = align_up(off + (size_t)P.BH * nseg * ((size_t)P.r * P.d + P.r) *
                             sizeof(float), 256);
    C->off_sB = off;
    off = align_up(off + (size_t)P.BH * nc * P.r * P.d * sizeof(uint16_t),
                   256);
    C->off_sA = off;
    off = align_up(off + (size_t)P.BH * nc * P.r * sizeof(float), 256);
    C->off_W = off;
    off = align_up(off + (size_t)P.H * P.Lg_pad * P.d * sizeof(uint16_t), 256);
    C->off_ctr = off;  // work counters of the attention launches
    off = align_up(off + (size_t)(Lv + 1) * sizeof(int), 256);
    C->total = off;
    return ELSAA_OK;
}

int causal_forward(const elsaa_params *params, const void *q, const void *k,
                   const void *v, const float *w_sort, const float *w_race,
                   const float *lambda_tok, const float *gates, void *o,
                   float *log_d_sparse, float *d_lr, float *m_sparse,
                   void *workspace, size_t workspace_bytes, void *stream) {
    CausalPlan C;
    const char *msg = "";
    int rc = make_causal_plan(params, &C, &msg);
    if (rc != ELSAA_OK) return fail(rc, "%s", msg);
    const Plan &P = C.P;
    if (!q || !k || !v || !o)
        return fail(ELSAA_ERR_INVALID_ARG, "q, k, v and o must be non-NULL");
    if (!w_race) return fail(ELSAA_ERR_INVALID_ARG, "w_race must be non-NULL");
    if (P.n_s > 0 && !w_sort)
        return fail(ELSAA_ERR_INVALID_ARG,
                    "w_sort must be non-NULL when sort_bits > 0");
    const void *ptrs[] = {q, k, v, o, w_race};
    for (const void *p : ptrs)
        if ((uintptr_t)p % 16)
            return fail(ELSAA_ERR_INVALID_ARG,
                        "q, k, v, o and w_race must be 16-byte aligned");
    if (gates && (uintptr_t)gates % 8)
        return fail(ELSAA_ERR_INVALID_ARG, "gates must be 8-byte aligned");
    if (!workspace) return fail(ELSAA_ERR_WORKSPACE, "workspace is NULL");
    if ((uintptr_t)workspace % 256)
        return fail(ELSAA_ERR_WORKSPACE, "workspace must be 256-byte aligned");
    if (workspace_bytes < C.total)
        return fail(ELSAA_ERR_WORKSPACE,
                    "workspace too small: %zu bytes given, %zu needed",
                    workspace_bytes, C.total);
    cudaStream_t st = (cudaStream_t)stream;
    char *ws = (char *)workspace;
    DeviceStatus *status = (DeviceStatus *)(ws + C.off_status);
    uint32_t *keyrank = (uint32_t *)(ws + C.off_keyrank);
    int *hist = (int *)(ws + C.off_hist);
    int32_t *perms = (int32_t *)(ws + C.off_perms);
    float *RO = (float *)(ws + C.off_RO);
    float *RL = (float *)(ws + C.off_RL);
    float *part = (float *)(ws + C.off_part);
    uint16_t *sB = (uint16_t *)(ws + C.off_sB);
    float *sA = (float *)(ws + C.off_sA);
    uint16_t *Wbf = (uint16_t *)(ws + C.off_W);
    int *ctr = (int *)(ws + C.off_ctr);

    ELSAA_CHECK_LAUNCH(cudaMemsetAsync(status, 0, sizeof(DeviceStatus), st),
                       "status reset");
    ELSAA_CHECK_LAUNCH(
        cudaMemsetAsync(ctr, 0, (size_t)(C.Lv + 1) * sizeof(int), st),
        "counter reset");
    // sparse branch: codes, sorted halves, base segments, then the levels
    ELSAA_CHECK_LAUNCH(timed("sort_hash", st, [&] {
                           return launch_sort_hash(P, q, k, w_sort, keyrank,
                                                   hist, status, st);
                       }),
                       "sort_hash");
    ELSAA_CHECK_LAUNCH(timed("seg_sort", st, [&] {
                           return launch_seg_sort(P, C.Lv, keyrank, perms,
                                                  st);
                       }),
                       "seg_sort");
    ELSAA_CHECK_LAUNCH(timed("causal_attn_base", st, [&] {
                           return launch_causal_attn(P, 0, C.n_leaf, 0, q, k,
                                                     v, perms, ctr, RO, RL,
                                                     status, st);
                       }),
                       "causal_attn_base");
    // the low-rank branch (chunk summaries, prefix states) on the side
    // stream from here: the base segments' persistent CTAs fill every SM
    // (all of TMEM), so these run beside the SortLSH levels instead of
    // delaying the sorts and the base segments
    SideStream *side = nullptr;
    ELSAA_CHECK_LAUNCH(side_stream(&side), "side stream");
    cudaStream_t ks = side->s;
    ELSAA_CHECK_LAUNCH(cudaEventRecord(side->fork, st), "fork");
    ELSAA_CHECK_LAUNCH(cudaStreamWaitEvent(ks, side->fork, 0), "fork wait");
    ELSAA_CHECK_LAUNCH(timed("prep_planes", ks, [&] {
                           return launch_prep_planes(P, w_race, Wbf, ks);
                       }),
                       "prep_planes");
    ELSAA_CHECK_LAUNCH(timed("race_keys_ws", ks, [&] {
                           return launch_race_keys_ws(C.Pc, k, v, Wbf, part,
                                                      status, ks);
                       }),
                       "race_keys_ws");
    ELSAA_CHECK_LAUNCH(timed("causal_scan", ks, [&] {
                           return launch_causal_scan(P, k, v, Wbf, part, sB,
                                                     sA, status, ks);
                       }),
                       "causal_scan");
    ELSAA_CHECK_LAUNCH(cudaEventRecord(side->join, ks), "join");
    for (int level = C.Lv; level >= 1; --level)
        ELSAA_CHECK_LAUNCH(timed("causal_attn_merge", st, [&] {
                               return launch_causal_attn(P, 1, C.n_leaf,
                                                         level, q, k, v,
                                                         perms, ctr + level,
                                                         RO, RL, status, st);
                           }),
                           "causal_attn_merge");
    ELSAA_CHECK_LAUNCH(cudaStreamWaitEvent(st, side->join, 0), "join wait");
    ELSAA_CHECK_LAUNCH(timed("causal_race", st, [&] {
                           return launch_causal_race(
                               P, q, k, v, Wbf, sB, sA, RO, RL, lambda_tok,
                               gates, o, log_d_sparse, d_lr, m_sparse, status,
                               st);
                       }),
                       "causal_race");
    return ELSAA_OK;
}

}  // namespace

extern "C" int elsaa_abi_version(void) { return ELSAA_ABI_VERSION; }

extern "C" const char *elsaa_last_error(void) { return g_err; }

extern "C" int elsaa_workspace_size(const elsaa_params *params,
                                    size_t *bytes) {
    g_err[0] = 0;
    if (!bytes) return fail(ELSAA_ERR_INVALID_ARG, "bytes is NULL");
    if (params && params->causal == 1) {
        CausalPlan C;
        const char *msg = "";
        int rc = make_causal_plan(params, &C, &msg);
        if (rc != ELSAA_OK) return fail(rc, "%s", msg);
        *bytes = C.total;
        return ELSAA_OK;
    }
    Plan P;
    const char *msg = "";
    int rc = make_plan(params, &P, &msg);
    if (rc != ELSAA_OK) return fail(rc, "%s", msg);
    *bytes = P.total;
    return ELSAA_OK;
}


namespace {

// The non-causal forward. gf: the gate network computed in the same call
// (its outputs are the gates / lambda_tok given here), or NULL.
int forward_impl(const elsaa_params *params, const void *q, const void *k,
                 const void *v, const float *w_sort, const float *w_race,
                 const float *lambda_tok, const float *gates, void *o,
                 float *log_d_sparse, float *d_lr, float *m_sparse,
                 int32_t *perm_q, int32_t *perm_k, void *workspace,
                 size_t workspace_bytes, void *stream,
                 const GateFusion *gf) {
    Plan P;
    const char *msg = "";
    int rc = make_plan(params, &P, &msg);
    if (rc != ELSAA_OK) return fail(rc, "%s", msg);
    if (!q || !k || !v || !o)
        return fail(ELSAA_ERR_INVALID_ARG, "q, k, v and o must be non-NULL");
    if (!w_race) return fail(ELSAA_ERR_INVALID_ARG, "w_race must be non-NULL");
    if (P.n_s > 0 && !w_sort)
        return fail(ELSAA_ERR_INVALID_ARG,
                    "w_sort must be non-NULL when sort_bits > 0");
    // rows are moved in 16-byte pieces (cp.async, vector loads)
    const void *ptrs[] = {q, k, v, o, w_race};
    for (const void *p : ptrs)
        if ((uintptr_t)p % 16)
            return fail(ELSAA_ERR_INVALID_ARG,
                        "q, k, v, o and w_race must be 16-byte aligned");
    if (!workspace)
        return fail(ELSAA_ERR_WORKSPACE, "workspace is NULL");
    if ((uintptr_t)workspace % 256)
        return fail(ELSAA_ERR_WORKSPACE, "workspace must be 256-byte aligned");
    if (workspace_bytes < P.total)
        return fail(ELSAA_ERR_WORKSPACE,
                    "workspace too small: %zu bytes given, %zu needed",
                    workspace_bytes, P.total);

    cudaStream_t st = (cudaStream_t)stream;
    char *ws = (char *)workspace;
    DeviceStatus *status = (DeviceStatus *)(ws + P.off_status);
    uint32_t *keyrank = (uint32_t *)(ws + P.off_keyrank);
    int *hist = (int *)(ws + P.off_hist);
    // the top-k selector keeps the sorted orders in the workspace (the
    // selected-key export reads them); the caller's copies follow
    int32_t *pq = perm_q && !P.sel ? perm_q : (int32_t *)(ws + P.off_perm);
    int32_t *pk = perm_k && !P.sel
                      ? perm_k
                      : (int32_t *)(ws + P.off_perm) + (size_t)P.BH * P.N;
    float *part = (float *)(ws + P.off_part);
    float *A = (float *)(ws + P.off_A);
    float *Bm = (float *)(ws + P.off_B);
    uint16_t *Bh = (uint16_t *)(ws + P.off_Bh);
    uint16_t *Wbf = (uint16_t *)(ws + P.off_W);

    ELSAA_CHECK_LAUNCH(cudaMemsetAsync(status, 0, sizeof(DeviceStatus), st),
                       "status reset");
    // RACE key side (no sort needed) on the side stream, launched first so
    // that its CTAs are placed before the hash kernel's
    SideStream *side = nullptr;
    ELSAA_CHECK_LAUNCH(side_stream(&side), "side stream");
    cudaStream_t ks = side->s;
    ELSAA_CHECK_LAUNCH(cudaEventRecord(side->fork, st), "fork");
    ELSAA_CHECK_LAUNCH(cudaStreamWaitEvent(ks, side->fork, 0), "fork wait");
    if (P.impl == 2) {
        ELSAA_CHECK_LAUNCH(timed("prep_planes", ks, [&] {
                               return launch_prep_planes(P, w_race, Wbf, ks);
                           }),
                           "prep_planes");
        ELSAA_CHECK_LAUNCH(timed("race_keys_ws", ks, [&] {
                               return launch_race_keys_ws(P, k, v, Wbf, part,
                                                          status, ks);
                           }),
                           "race_keys_ws");
    } else {
        ELSAA_CHECK_LAUNCH(timed("race_partial_simt", ks, [&] {
                               return launch_race_partial_simt(P, k, v, w_race,
                                                               part, ks);
                           }),
                           "race_partial_simt");
    }
    ELSAA_CHECK_LAUNCH(timed("race_reduce", ks, [&] {
                           return launch_race_reduce(P, part, A, Bm, Bh, ks);
                       }),
                       "race_reduce");
    ELSAA_CHECK_LAUNCH(cudaEventRecord(side->join, ks), "join");
    ELSAA_CHECK_LAUNCH(timed("sort_hash", st, [&] {
                           return launch_sort_hash(P, q, k, w_sort, keyrank,
                                                   hist, status, st);
                       }),
                       "sort_hash");
    ELSAA_CHECK_LAUNCH(timed("sort_scan", st,
                             [&] { return launch_sort_scan(P, hist, st); }),
                       "sort_scan");
    ELSAA_CHECK_LAUNCH(timed("sort_scatter", st, [&] {
                           return launch_sort_scatter(P, keyrank, hist, pq,
                                                      pk, status, st);
                       }),
                       "sort_scatter");
    // the gate network (elsaa_forward_gated): on the caller's stream right
    // after the sort, so its CTAs take the SMs that the sort chain leaves
    // idle while the RACE key side (the longer chain) finishes
    if (gf)
        ELSAA_CHECK_LAUNCH(timed("gate_mlp", st, [&] {
                               return launch_gates(P, *gf->mlp, q, gf->gates,
                                                   gf->lam, gf->gate_ws,
                                                   status, st);
                           }),
                           "gate_mlp");
    int32_t *cand = nullptr;
    uint32_t *selmask = nullptr;
    if (P.sel) {
        cand = (int32_t *)(ws + P.off_cand);
        selmask = (uint32_t *)(ws + P.off_mask);
        static const char *const kStage[3] = {"topk_sums", "topk_cand",
                                              "topk_select"};
        for (int sg = 0; sg < 3; ++sg)
            ELSAA_CHECK_LAUNCH(timed(kStage[sg], st, [&] {
                                   return launch_topk(
                                       sg, P, q, k, pq, pk,
                                       (float *)(ws + P.off_sums), cand,
                                       selmask, status, st);
                               }),
                               kStage[sg]);
        const size_t pb = (size_t)P.BH * P.N * sizeof(int32_t);
        if (perm_q)
            ELSAA_CHECK_LAUNCH(cudaMemcpyAsync(perm_q, pq, pb,
                                               cudaMemcpyDeviceToDevice, st),
                               "copy of perm_q");
        if (perm_k)
            ELSAA_CHECK_LAUNCH(cudaMemcpyAsync(perm_k, pk, pb,
                                               cudaMemcpyDeviceToDevice, st),
                               "copy of perm_k");
    }
    ELSAA_CHECK_LAUNCH(cudaStreamWaitEvent(st, side->join, 0), "join wait");
    // neighbouring key blocks (nb > 0) run in the persistent kernel for
    // b of 128 or 256 and nb = 1, otherwise in the CUDA-core block kernel;
    // the RACE key side above does not depend on them
    if (P.impl == 2 && pair_supported(P)) {
        // key blocks of 256: the two query tiles of a block on a CTA pair
        ELSAA_CHECK_LAUNCH(timed("block_attn_pair", st, [&] {
                               return launch_block_attn_pair(
                                   P, q, k, v, Wbf, pq, pk, A, Bh,
                                   lambda_tok, gates, o, log_d_sparse, d_lr,
                                   m_sparse, status, st);
                           }),
                           "block_attn_pair");
    } else if (P.impl == 2 && ws_supported(P)) {
        ELSAA_CHECK_LAUNCH(timed("block_attn_ws", st, [&] {
                               return launch_block_attn_ws(
                                   P, q, k, v, Wbf, pq, pk, A, Bh,
                                   lambda_tok, gates, o, log_d_sparse, d_lr,
                                   m_sparse, status, st, cand, selmask);
                           }),
                           "block_attn_ws");
    } else {
        ELSAA_CHECK_LAUNCH(timed("block_attn_simt", st, [&] {
                               return launch_block_attn_simt(
                                   P, q, k, v, w_race, pq, pk, A, Bm,
                                   lambda_tok, gates, o, log_d_sparse, d_lr,
                                   m_sparse, status, st, cand, selmask);
                           }),
                           "block_attn_simt");
    }
    return ELSAA_OK;
}

}  // namespace

extern "C" int elsaa_forward(const elsaa_params *params, const void *q,
                             const void *k, const void *v,
                             const float *w_sort, const float *w_race,
                             const float *lambda_tok, const float *gates,
                             void *o, float *log_d_sparse, float *d_lr,
                             float *m_sparse, int32_t *perm_q,
                             int32_t *perm_k, void *workspace,
                             size_t workspace_bytes, void *stream) {
    g_err[0] = 0;
    if (params && params->causal == 1)
        return causal_forward(params, q, k, v, w_sort, w_race, lambda_tok,
                              gates, o, log_d_sparse, d_lr, m_sparse,
                              workspace, workspace_bytes, stream);
    return forward_impl(params, q, k, v, w_sort, w_race, lambda_tok, gates,
                        o, log_d_sparse, d_lr, m_sparse, perm_q, perm_k,
                        workspace, workspace_bytes, stream, nullptr);
}

// ---------------------------------------------------------------- backward

namespace {

// Backward workspace: status | RACE chunk partials (A, B, then gA, gB) |
// A | B | gA | gB | gNum / L [B*H][N][d_h] | gDen / L [B*H][N] | bf16
// planes | bf16 B | bf16 gB. The tensor-core path sums gA, gB inside the
// block kernel: it has no gNum / gDen arrays.
struct BwdPlan {
    Plan P;    // forward geometry with CUDA-core RACE chunking
    Plan Pf;   // the forward's own plan (tensor-core key summaries if bf16)
    size_t off_status, off_part, off_A, off_B, off_gA, off_gB, off_gnum,
        off_gden, off_W, off_Bh, total;
    bool tc;   // tensor-core block kernel (bf16 operands)
};

int make_bwd_plan(const elsaa_params *p, BwdPlan *Bp, const char **msg) {
    if (p && p->causal) {
        *msg = "elsaa_backward: the causal variant has no backward pass here";
        return ELSAA_ERR_UNSUPPORTED;
    }
    if (p && p->selector != 0) {
        *msg = "elsaa_backward: built for the sorted-block selector only";
        return ELSAA_ERR_UNSUPPORTED;
    }
    elsaa_params q = *p;
    q.impl = ELSAA_IMPL_SIMT;  // the backward runs on CUDA cores
    int rc = make_plan(&q, &Bp->P, msg);
    if (rc != ELSAA_OK) return rc;
    if (Bp->P.nb != 0) {
        *msg = "elsaa_backward requires neighbor_blocks = 0";
        return ELSAA_ERR_UNSUPPORTED;
    }
    rc = make_plan(p, &Bp->Pf, msg);  // A, B as the forward makes them
    if (rc != ELSAA_OK) return rc;
    const Plan &P = Bp->P;
    // the tensor-core kernels read B and write gB as bf16
    Bp->tc = p->impl == ELSAA_IMPL_AUTO && Bp->Pf.impl == 2 &&
             bwd_tc_supported(Bp->Pf);
    int S = P.S > Bp->Pf.S ? P.S : Bp->Pf.S;
    if (Bp->tc && bwd_tc_segments(Bp->Pf) > S) S = bwd_tc_segments(Bp->Pf);
    if (!bwd_supported(P)) {
        *msg = "backward: this block size, d_h and r need more shared "
               "memory than an SM has";
        return ELSAA_ERR_UNSUPPORTED;
    }
    const size_t BHN = (size_t)P.BH * P.N;
    const size_t per = (size_t)P.r * P.d + P.r;
    size_t off = 0;
    Bp->off_status = off;
    off = align_up(off + sizeof(DeviceStatus), 256);
    Bp->off_part = off;
    off = align_up(off + (size_t)P.BH * S * per * sizeof(float), 256);
    Bp->off_A = off;
    off = align_up(off + (size_t)P.BH * P.r * sizeof(float), 256);
    Bp->off_B = off;
    off = align_up(off + (size_t)P.BH * P.r * P.d * sizeof(float), 256);
    Bp->off_gA = off;  // gA, gB: CUDA-core path (the tensor-core key
                       // kernel sums the partials itself)
    if (!Bp->tc) off = align_up(off + (size_t)P.BH * P.r * sizeof(float), 256);
    Bp->off_gB = off;
    if (!Bp->tc)
        off = align_up(off + (size_t)P.BH * P.r * P.d * sizeof(float), 256);
    Bp->off_gnum = off;
    if (!Bp->tc) off = align_up(off + BHN * P.d * sizeof(float), 256);
    Bp->off_gden = off;
    if (!Bp->tc) off = align_up(off + BHN * sizeof(float), 256);
    Bp->off_W = off;
    off = align_up(off + (size_t)P.H * P.Lg_pad * P.d * sizeof(uint16_t), 256);
    Bp->off_Bh = off;
    if (Bp->tc)
        off = align_up(off + (size_t)P.BH * P.r * P.d * sizeof(uint16_t),
                       256);
    Bp->total = off;
    return ELSAA_OK;
}

}  // namespace

extern "C" int elsaa_forward_race_summaries(const elsaa_params *params,
                                            const void *workspace,
                                            size_t workspace_bytes,
                                            float *race_A, float *race_B,
                                            void *stream) {
    g_err[0] = 0;
    if (params && params->causal == 1)
        return fail(ELSAA_ERR_UNSUPPORTED,
                    "the causal forward keeps per-chunk prefix states, not "
                    "whole-sequence summaries");
    Plan P;
    const char *msg = "";
    int rc = make_plan(params, &P, &msg);
    if (rc != ELSAA_OK) return fail(rc, "%s", msg);
    if (!race_A || !race_B)
        return fail(ELSAA_ERR_INVALID_ARG, "race_A and race_B must be non-NULL");
    if (!workspace) return fail(ELSAA_ERR_WORKSPACE, "workspace is NULL");
    if (workspace_bytes < P.total)
        return fail(ELSAA_ERR_WORKSPACE,
                    "workspace too small: %zu bytes given, %zu needed",
                    workspace_bytes, P.total);
    cudaStream_t st = (cudaStream_t)stream;
    const char *ws = (const char *)workspace;
    ELSAA_CHECK_LAUNCH(
        cudaMemcpyAsync(race_A, ws + P.off_A,
                        (size_t)P.BH * P.r * sizeof(float),
                        cudaMemcpyDeviceToDevice, st),
        "copy of A");
    ELSAA_CHECK_LAUNCH(
        cudaMemcpyAsync(race_B, ws + P.off_B,
                        (size_t)P.BH * P.r * P.d * sizeof(float),
                        cudaMemcpyDeviceToDevice, st),
        "copy of B");
    return ELSAA_OK;
}

extern "C" int elsaa_forward_selected_keys(const elsaa_params *params,
                                           const void *workspace,
                                           size_t workspace_bytes,
                                           int32_t *keys, void *stream) {
    g_err[0] = 0;
    if (!params || params->selector != 1)
        return fail(ELSAA_ERR_INVALID_ARG, "params must have selector = 1");
    Plan P;
    const char *msg = "";
    int rc = make_plan(params, &P, &msg);
    if (rc != ELSAA_OK) return fail(rc, "%s", msg);
    if (!keys) return fail(ELSAA_ERR_INVALID_ARG, "keys is NULL");
    if (!workspace) return fail(ELSAA_ERR_WORKSPACE, "workspace is NULL");
    if (workspace_bytes < P.total)
        return fail(ELSAA_ERR_WORKSPACE,
                    "workspace too small: %zu bytes given, %zu needed",
                    workspace_bytes, P.total);
    char *ws = (char *)workspace;
    const int32_t *pq = (const int32_t *)(ws + P.off_perm);
    ELSAA_CHECK_LAUNCH(
        launch_topk_export(P, pq, pq + (size_t)P.BH * P.N,
                           (const int32_t *)(ws + P.off_cand),
                           (const uint32_t *)(ws + P.off_mask), keys,
                           (DeviceStatus *)(ws + P.off_status),
                           (cudaStream_t)stream),
        "topk_export");
    return ELSAA_OK;
}

extern "C" int elsaa_causal_levels(const elsaa_params *params,
                                   int *levels) {
    g_err[0] = 0;
    if (!levels) return fail(ELSAA_ERR_INVALID_ARG, "levels is NULL");
    if (!params || params->causal != 1)
        return fail(ELSAA_ERR_INVALID_ARG, "params must have causal = 1");
    CausalPlan C;
    const char *msg = "";
    int rc = make_causal_plan(params, &C, &msg);
    if (rc != ELSAA_OK) return fail(rc, "%s", msg);
    *levels = C.Lv;
    return ELSAA_OK;
}

extern "C" int elsaa_causal_index_lists(const elsaa_params *params,
                                        const void *workspace,
                                        size_t workspace_bytes,
                                        int32_t *lists, void *stream) {
    g_err[0] = 0;
    if (!params || params->causal != 1)
        return fail(ELSAA_ERR_INVALID_ARG, "params must have causal = 1");
    CausalPlan C;
    const char *msg = "";
    int rc = make_causal_plan(params, &C, &msg);
    if (rc != ELSAA_OK) return fail(rc, "%s", msg);
    if (C.Lv == 0) return ELSAA_OK;  // one segment: nothing is sorted
    if (!lists) return fail(ELSAA_ERR_INVALID_ARG, "lists is NULL");
    if (!workspace) return fail(ELSAA_ERR_WORKSPACE, "workspace is NULL");
    if (workspace_bytes < C.total)
        return fail(ELSAA_ERR_WORKSPACE,
                    "workspace too small: %zu bytes given, %zu needed",
                    workspace_bytes, C.total);
    const char *ws = (const char *)workspace;
    ELSAA_CHECK_LAUNCH(
        cudaMemcpyAsync(lists, ws + C.off_perms,
                        (size_t)C.Lv * C.P.BH * C.P.N * sizeof(int32_t),
                        cudaMemcpyDeviceToDevice, (cudaStream_t)stream),
        "copy of the index lists");
    return ELSAA_OK;
}

extern "C" int elsaa_backward_workspace_size(const elsaa_params *params,
                                             size_t *bytes) {
    g_err[0] = 0;
    if (!bytes) return fail(ELSAA_ERR_INVALID_ARG, "bytes is NULL");
    BwdPlan Bp;
    const char *msg = "";
    int rc = make_bwd_plan(params, &Bp, &msg);
    if (rc != ELSAA_OK) return fail(rc, "%s", msg);
    *bytes = Bp.total;
    return ELSAA_OK;
}

extern "C" int elsaa_backward(const elsaa_params *params, const void *q,
                              const void *k, const void *v,
                              const float *w_sort, const float *w_race,
                              const float *lambda_tok, const float *gates,
                              const void *d_o, const int32_t *perm_q,
                              const int32_t *perm_k, float *dq, float *dk,
                              float *dv, float *d_gates, float *d_lambda,
                              const float *race_A, const float *race_B,
                              void *workspace, size_t workspace_bytes,
                              void *stream) {
    (void)w_sort;  // the permutations are given
    g_err[0] = 0;
    BwdPlan Bp;
    const char *msg = "";
    int rc = make_bwd_plan(params, &Bp, &msg);
    if (rc != ELSAA_OK) return fail(rc, "%s", msg);
    const Plan &P = Bp.P;
    if (!q || !k || !v || !d_o || !dq || !dk || !dv)
        return fail(ELSAA_ERR_INVALID_ARG,
                    "q, k, v, d_o, dq, dk and dv must be non-NULL");
    if (!w_race) return fail(ELSAA_ERR_INVALID_ARG, "w_race must be non-NULL");
    if (!perm_q || !perm_k)
        return fail(ELSAA_ERR_INVALID_ARG,
                    "perm_q and perm_k (from elsaa_forward) are required");
    const void *ptrs[] = {q, k, v, d_o, w_race, dq, dk, dv};
    for (const void *p : ptrs)
        if ((uintptr_t)p % 16)
            return fail(ELSAA_ERR_INVALID_ARG,
                        "q, k, v, d_o, w_race, dq, dk and dv must be 16-byte "
                        "aligned");
    if ((race_A == nullptr) != (race_B == nullptr))
        return fail(ELSAA_ERR_INVALID_ARG,
                    "race_A and race_B must be given together");
    if ((uintptr_t)race_A % 16 || (uintptr_t)race_B % 16)
        return fail(ELSAA_ERR_INVALID_ARG,
                    "race_A and race_B must be 16-byte aligned");
    if (!workspace) return fail(ELSAA_ERR_WORKSPACE, "workspace is NULL");
    if ((uintptr_t)workspace % 256)
        return fail(ELSAA_ERR_WORKSPACE, "workspace must be 256-byte aligned");
    if (workspace_bytes < Bp.total)
        return fail(ELSAA_ERR_WORKSPACE,
                    "workspace too small: %zu bytes given, %zu needed",
                    workspace_bytes, Bp.total);

    cudaStream_t st = (cudaStream_t)stream;
    char *ws = (char *)workspace;
    DeviceStatus *status = (DeviceStatus *)(ws + Bp.off_status);
    float *part = (float *)(ws + Bp.off_part);
    float *A = (float *)(ws + Bp.off_A);
    float *Bm = (float *)(ws + Bp.off_B);
    float *gA = (float *)(ws + Bp.off_gA);
    float *gB = (float *)(ws + Bp.off_gB);
    float *gnum = (float *)(ws + Bp.off_gnum);
    float *gden = (float *)(ws + Bp.off_gden);

    ELSAA_CHECK_LAUNCH(cudaMemsetAsync(status, 0, sizeof(DeviceStatus), st),
                       "status reset");
    // A, B: the forward's saved summaries, or recomputed exactly as the
    // forward made them
    const Plan &Pf = Bp.Pf;
    uint16_t *Wbf = (uint16_t *)(ws + Bp.off_W);
    uint16_t *Bhw = Bp.tc ? (uint16_t *)(ws + Bp.off_Bh) : nullptr;
    const size_t nB = (size_t)P.BH * P.r * P.d;
    // the bf16 planes and, with saved summaries, the bf16 image of B: one
    // launch where both are needed
    const bool images = Pf.impl == 2 && race_A && Bhw && nB % 4 == 0;
    if (images)
        ELSAA_CHECK_LAUNCH(timed("planes_and_image", st, [&] {
                               return launch_planes_and_image(
                                   Pf, w_race, Wbf, race_B, Bhw, nB, st);
                           }),
                           "planes_and_image");
    else if (Pf.impl == 2)
        ELSAA_CHECK_LAUNCH(timed("prep_planes", st, [&] {
                               return launch_prep_planes(Pf, w_race, Wbf, st);
                           }),
                           "prep_planes");
    if (race_A) {
        A = const_cast<float *>(race_A);
        Bm = const_cast<float *>(race_B);
        if (Bhw && !images)
            ELSAA_CHECK_LAUNCH(timed("bf16_image", st, [&] {
                                   return launch_bf16_image(race_B, Bhw, nB,
                                                            st);
                               }),
                               "bf16_image");
    } else {
        if (Pf.impl == 2) {
            ELSAA_CHECK_LAUNCH(timed("race_keys_ws", st, [&] {
                                   return launch_race_keys_ws(
                                       Pf, k, v, Wbf, part, status, st);
                               }),
                               "race_keys_ws");
        } else {
            ELSAA_CHECK_LAUNCH(timed("race_partial_simt", st, [&] {
                                   return launch_race_partial_simt(
                                       Pf, k, v, w_race, part, st);
                               }),
                               "race_partial_simt");
        }
        ELSAA_CHECK_LAUNCH(timed("race_reduce", st, [&] {
                               return launch_race_reduce(Pf, part, A, Bm,
                                                         Bhw, st);
                           }),
                           "race_reduce");
    }
    if (Bp.tc) {
        ELSAA_CHECK_LAUNCH(timed("bwd_block_tc", st, [&] {
                               return launch_bwd_block_tc(
                                   Pf, q, k, v, d_o,
                                   (const uint16_t *)(ws + Bp.off_W), Bhw, A,
                                   perm_q, perm_k, lambda_tok, gates, dq, dk,
                                   dv, d_gates, d_lambda, part, status, st);
                           }),
                           "bwd_block_tc");
    } else {
        ELSAA_CHECK_LAUNCH(timed("bwd_block", st, [&] {
                               return launch_bwd_block(
                                   P, q, k, v, d_o, w_race, A, Bm, perm_q,
                                   perm_k, lambda_tok, gates, dq, dk, dv,
                                   d_gates, d_lambda, gnum, gden, status,
                                   st);
                           }),
                           "bwd_block");
    }
    if (!Bp.tc) {
        ELSAA_CHECK_LAUNCH(timed("bwd_race_sums", st, [&] {
                               return launch_race_partial_weighted(
                                   P, q, gnum, gden, w_race, part, st);
                           }),
                           "bwd_race_sums");
        ELSAA_CHECK_LAUNCH(timed("race_reduce", st, [&] {
                               return launch_race_reduce(P, part, gA, gB,
                                                         nullptr, st);
                           }),
                           "race_reduce");
    }
    if (Bp.tc) {
        ELSAA_CHECK_LAUNCH(timed("bwd_keys_tc", st, [&] {
                               return launch_bwd_keys_tc(
                                   Pf, k, v,
                                   (const uint16_t *)(ws + Bp.off_W), part, dk,
                                   dv, status, st);
                           }),
                           "bwd_keys_tc");
    } else {
        ELSAA_CHECK_LAUNCH(timed("bwd_keys", st, [&] {
                               return launch_bwd_keys(P, k, v, w_race, gA, gB,
                                                      dk, dv, st);
                           }),
                           "bwd_keys");
    }
    return ELSAA_OK;
}

namespace {

// Validates the gate MLP description for the (already planned) shapes.
int check_gate_mlp(const elsaa_gate_mlp *m, const char **msg) {
    if (!m) {
        *msg = "mlp is NULL";
        return ELSAA_ERR_INVALID_ARG;
    }
    if (m->hidden < 16 || m->hidden > 128 || m->hidden % 16) {
        *msg = "mlp->hidden must be a multiple of 16 in [16, 128]";
        return ELSAA_ERR_UNSUPPORTED;
    }
    if (!m->w1 || !m->b1 || !m->w2 || !m->b2) {
        *msg = "mlp->w1, b1, w2 and b2 must be non-NULL";
        return ELSAA_ERR_INVALID_ARG;
    }
    if (m->w_lambda && (!m->b_lambda || !m->c_lambda)) {
        *msg = "mlp->b_lambda and c_lambda are required with w_lambda";
        return ELSAA_ERR_INVALID_ARG;
    }
    if (m->w_lambda && !(m->lambda_min > 0.0f)) {
        *msg = "mlp->lambda_min must be > 0";
        return ELSAA_ERR_INVALID_ARG;
    }
    return ELSAA_OK;
}

}  // namespace

extern "C" int elsaa_gates_workspace_size(const elsaa_params *params,
                                          const elsaa_gate_mlp *mlp,
                                          size_t *bytes) {
    g_err[0] = 0;
    if (!bytes) return fail(ELSAA_ERR_INVALID_ARG, "bytes is NULL");
    Plan P;
    const char *msg = "";
    int rc = make_plan(params, &P, &msg);
    if (rc == ELSAA_OK) rc = check_gate_mlp(mlp, &msg);
    if (rc != ELSAA_OK) return fail(rc, "%s", msg);
    *bytes = gate_workspace_bytes(P, mlp->hidden);
    return ELSAA_OK;
}

extern "C" int elsaa_gates(const elsaa_params *params,
                           const elsaa_gate_mlp *mlp, const void *q,
                           float *gates, float *lambda_tok, void *workspace,
                           size_t workspace_bytes, void *stream) {
    g_err[0] = 0;
    Plan P;
    const char *msg = "";
    int rc = make_plan(params, &P, &msg);
    if (rc == ELSAA_OK) rc = check_gate_mlp(mlp, &msg);
    if (rc != ELSAA_OK) return fail(rc, "%s", msg);
    if (!q || !gates)
        return fail(ELSAA_ERR_INVALID_ARG, "q and gates must be non-NULL");
    if (mlp->w_lambda && !lambda_tok)
        return fail(ELSAA_ERR_INVALID_ARG,
                    "lambda_tok must be non-NULL when mlp->w_lambda is given");
    if ((uintptr_t)q % 16 || (uintptr_t)gates % 8 ||
        (uintptr_t)mlp->b1 % 16 || (uintptr_t)mlp->w2 % 16)
        return fail(ELSAA_ERR_INVALID_ARG,
                    "q, mlp->b1 and mlp->w2 must be 16-byte and gates 8-byte "
                    "aligned");
    const size_t need = gate_workspace_bytes(P, mlp->hidden);
    if (!workspace) return fail(ELSAA_ERR_WORKSPACE, "workspace is NULL");
    if ((uintptr_t)workspace % 256)
        return fail(ELSAA_ERR_WORKSPACE, "workspace must be 256-byte aligned");
    if (workspace_bytes < need)
        return fail(ELSAA_ERR_WORKSPACE,
                    "workspace too small: %zu bytes given, %zu needed",
                    workspace_bytes, need);
    cudaStream_t st = (cudaStream_t)stream;
    char *ws = (char *)workspace;
    DeviceStatus *status = (DeviceStatus *)ws;
    uint16_t *wbf = (uint16_t *)(ws + 256);
    ELSAA_CHECK_LAUNCH(cudaMemsetAsync(status, 0, sizeof(DeviceStatus), st),
                       "status reset");
    ELSAA_CHECK_LAUNCH(timed("gate_mlp", st, [&] {
                           return launch_gates(P, *mlp, q, gates,
                                               mlp->w_lambda ? lambda_tok
                                                             : nullptr,
                                               wbf, status, st);
                       }),
                       "gate_mlp");
    return ELSAA_OK;
}

namespace {

// Extra workspace of elsaa_forward_gated after the forward's own: the gate
// kernel's workspace (elsaa_gates' layout), then the gates [B*H*N][2] and
// lambda [B*H*N] (fp32).
struct GatedPlan {
    size_t fwd, off_gws, off_gates, off_lam, total;
};

int make_gated_plan(const elsaa_params *params, const elsaa_gate_mlp *mlp,
                    GatedPlan *G, const char **msg) {
    static thread_local char fwd_msg[256];
    size_t fwd = 0;
    int rc = elsaa_workspace_size(params, &fwd);
    if (rc != ELSAA_OK) {
        snprintf(fwd_msg, sizeof(fwd_msg), "%s", elsaa_last_error());
        *msg = fwd_msg;
        return rc;
    }
    Plan P;
    rc = make_plan(params, &P, msg);
    if (rc == ELSAA_OK) rc = check_gate_mlp(mlp, msg);
    if (rc != ELSAA_OK) return rc;
    size_t off = align_up(fwd, 256);
    G->fwd = fwd;
    G->off_gws = off;
    off = align_up(off + gate_workspace_bytes(P, mlp->hidden), 256);
    const size_t BHN = (size_t)P.BH * P.N;
    G->off_gates = off;
    off = align_up(off + BHN * 2 * sizeof(float), 256);
    G->off_lam = off;
    off = align_up(off + BHN * sizeof(float), 256);
    G->total = off;
    return ELSAA_OK;
}

}  // namespace

extern "C" int elsaa_forward_gated_workspace_size(const elsaa_params *params,
                                                  const elsaa_gate_mlp *mlp,
                                                  size_t *bytes) {
    g_err[0] = 0;
    if (!bytes) return fail(ELSAA_ERR_INVALID_ARG, "bytes is NULL");
    GatedPlan G;
    const char *msg = "";
    int rc = make_gated_plan(params, mlp, &G, &msg);
    if (rc != ELSAA_OK) return fail(rc, "%s", msg);
    *bytes = G.total;
    return ELSAA_OK;
}

extern "C" int elsaa_forward_gated(
    const elsaa_params *params, const elsaa_gate_mlp *mlp, const void *q,
    const void *k, const void *v, const float *w_sort, const float *w_race,
    void *o, float *log_d_sparse, float *d_lr, float *m_sparse,
    int32_t *perm_q, int32_t *perm_k, float *gates_out, float *lambda_out,
    void *workspace, size_t workspace_bytes, void *stream) {
    g_err[0] = 0;
    GatedPlan G;
    const char *msg = "";
    int rc = make_gated_plan(params, mlp, &G, &msg);
    if (rc != ELSAA_OK) return fail(rc, "%s", msg);
    if (!q) return fail(ELSAA_ERR_INVALID_ARG, "q must be non-NULL");
    if ((uintptr_t)q % 16 || (uintptr_t)mlp->b1 % 16 ||
        (uintptr_t)mlp->w2 % 16 || (gates_out && (uintptr_t)gates_out % 8))
        return fail(ELSAA_ERR_INVALID_ARG,
                    "q, mlp->b1 and mlp->w2 must be 16-byte and gates_out "
                    "8-byte aligned");
    if (!workspace) return fail(ELSAA_ERR_WORKSPACE, "workspace is NULL");
    if ((uintptr_t)workspace % 256)
        return fail(ELSAA_ERR_WORKSPACE, "workspace must be 256-byte aligned");
    if (workspace_bytes < G.total)
        return fail(ELSAA_ERR_WORKSPACE,
                    "workspace too small: %zu bytes given, %zu needed",
                    workspace_bytes, G.total);
    cudaStream_t st = (cudaStream_t)stream;
    char *ws = (char *)workspace;
    float *gts = gates_out ? gates_out : (float *)(ws + G.off_gates);
    float *lam = mlp->w_lambda
                     ? (lambda_out ? lambda_out : (float *)(ws + G.off_lam))
                     : nullptr;
    if (params->causal) {
        // causal: the gate kernel of elsaa_gates, then the forward
        rc = elsaa_gates(params, mlp, q, gts, lam, ws + G.off_gws,
                         G.off_gates - G.off_gws, stream);
        if (rc != ELSAA_OK) return rc;
        return elsaa_forward(params, q, k, v, w_sort, w_race, lam, gts, o,
                             log_d_sparse, d_lr, m_sparse, perm_q, perm_k,
                             workspace, G.fwd, stream);
    }
    GateFusion gf;
    gf.mlp = mlp;
    gf.gate_ws = (uint16_t *)(ws + G.off_gws + 256);
    gf.gates = gts;
    gf.lam = lam;
    return forward_impl(params, q, k, v, w_sort, w_race, lam, gts, o,
                        log_d_sparse, d_lr, m_sparse, perm_q, perm_k,
                        workspace, G.fwd, stream, &gf);
}

extern "C" int elsaa_selftest_wait_timeout(void *workspace,
                                           size_t workspace_bytes,
                                           int limit_ms, void *stream) {
    g_err[0] = 0;
    if (!workspace || workspace_bytes < sizeof(DeviceStatus))
        return fail(ELSAA_ERR_WORKSPACE, "workspace missing or too small");
    if ((uintptr_t)workspace % 256)
        return fail(ELSAA_ERR_WORKSPACE, "workspace must be 256-byte aligned");
    if (limit_ms < 1 || limit_ms > 2000)
        return fail(ELSAA_ERR_INVALID_ARG, "limit_ms must be in [1, 2000]");
    cudaStream_t st = (cudaStream_t)stream;
    DeviceStatus *status = (DeviceStatus *)workspace;
    ELSAA_CHECK_LAUNCH(cudaMemsetAsync(status, 0, sizeof(DeviceStatus), st),
                       "status reset");
    ELSAA_CHECK_LAUNCH(launch_selftest_wait(status, limit_ms, st),
                       "selftest_wait");
    return ELSAA_OK;
}

extern "C" int elsaa_check_status(const void *workspace, void *stream) {
    g_err[0] = 0;
    if (!workspace) return fail(ELSAA_ERR_INVALID_ARG, "workspace is NULL");
    cudaStream_t st = (cudaStream_t)stream;
    cudaError_t e = cudaStreamSynchronize(st);
    if (e != cudaSuccess)
        return fail(ELSAA_ERR_CUDA, "stream: %s", cudaGetErrorString(e));
    DeviceStatus s;
    e = cudaMemcpy(&s, workspace, sizeof(s), cudaMemcpyDeviceToHost);
    if (e != cudaSuccess)
        return fail(ELSAA_ERR_CUDA, "status read: %s", cudaGetErrorString(e));
    if (s.code != 0)
        return fail(ELSAA_ERR_DEVICE,
                    "device status %d at site %d (info %d, %d)", s.code,
                    s.where, s.info0, s.info1);
    return ELSAA_OK;
}

extern "C" int elsaa_profile_start(void) {
    std::lock_guard<std::mutex> lk(g_prof_mu);
    g_prof_on = true;
    return ELSAA_OK;
}

extern "C" int elsaa_profile_stop(elsaa_kernel_stat *out, int max_entries,
                                  int *n_entries) {
    g_err[0] = 0;
    std::lock_guard<std::mutex> lk(g_prof_mu);
    g_prof_on = false;
    std::vector<std::string> names;
    std::vector<int> counts;
    std::vector<double> ms;
    int rc = ELSAA_OK;
    for (auto &r : g_prof) {
        float t = 0.f;
        cudaError_t e = cudaEventSynchronize(r.b);
        if (e == cudaSuccess) e = cudaEventElapsedTime(&t, r.a, r.b);
        if (e != cudaSuccess && rc == ELSAA_OK)
            rc = fail(ELSAA_ERR_CUDA, "profile: %s", cudaGetErrorString(e));
        size_t i = 0;
        while (i < names.size() && names[i] != r.name) ++i;
        if (i == names.size()) {
            names.push_back(r.name);
            counts.push_back(0);
            ms.push_back(0.0);
        }
        counts[i] += 1;
        ms[i] += t;
        g_ev_pool.push_back(r.a);
        g_ev_pool.push_back(r.b);
    }
    g_prof.clear();
    int n = 0;
    for (size_t i = 0; i < names.size() && (int)i < max_entries; ++i, ++n) {
        if (!out) break;
        snprintf(out[i].name, sizeof(out[i].name), "%s", names[i].c_str());
        out[i].launches = counts[i];
        out[i].total_ms = ms[i];
    }
    if (n_entries) *n_entries = out ? n : (int)names.size();
    return rc;
}
