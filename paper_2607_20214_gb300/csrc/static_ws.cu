// elsaa_forward_noalloc and its companions: the forward pass with scratch
// taken from a fixed array in the library's device image, for callers that
// cannot allocate device memory (see include/elsaa.h for the contract).
#include "internal.h"

namespace {

// The scratch array. In host code this name is only a host-side handle for
// the device symbol, never a device address: its device address is looked
// up with cudaGetSymbolAddress below.
static __device__ __align__(256) unsigned char
    g_static_workspace[ELSAA_STATIC_WORKSPACE_BYTES];

// Device address of the array on the current device. Looked up on every
// call (a cheap query that allocates nothing), so a device reset or a new
// primary context, which reloads the module at another address, never
// leaves a stale pointer behind.
int static_workspace(void **ptr) {
    void *p = nullptr;
    cudaError_t e = cudaGetSymbolAddress(&p, g_static_workspace);
    if (e != cudaSuccess || !p)
        return elsaa::set_last_error(ELSAA_ERR_CUDA,
                                     "cudaGetSymbolAddress: %s",
                                     cudaGetErrorString(e));
    *ptr = p;
    return ELSAA_OK;
}

}  // namespace

extern "C" int elsaa_forward_noalloc(const elsaa_params *params,
                                     const void *q, const void *k,
                                     const void *v, const float *w_sort,
                                     const float *w_race,
                                     const float *lambda_tok,
                                     const float *gates, void *o,
                                     float *log_d_sparse, float *d_lr,
                                     float *m_sparse, int32_t *perm_q,
                                     int32_t *perm_k, void *stream) {
    size_t need = 0;
    int rc = elsaa_workspace_size(params, &need);
    if (rc != ELSAA_OK) return rc;
    if (need > ELSAA_STATIC_WORKSPACE_BYTES)
        return elsaa::set_last_error(
            ELSAA_ERR_WORKSPACE,
            "problem needs %zu bytes of scratch; the static array of "
            "elsaa_forward_noalloc holds %zu",
            need, (size_t)ELSAA_STATIC_WORKSPACE_BYTES);
    void *ws = nullptr;
    rc = static_workspace(&ws);
    if (rc != ELSAA_OK) return rc;
    return elsaa_forward(params, q, k, v, w_sort, w_race, lambda_tok, gates,
                         o, log_d_sparse, d_lr, m_sparse, perm_q, perm_k, ws,
                         ELSAA_STATIC_WORKSPACE_BYTES, stream);
}

// The status word of the forward pass sits at the start of its workspace,
// here the start of the static array.
extern "C" int elsaa_check_status_noalloc(void *stream) {
    void *ws = nullptr;
    int rc = static_workspace(&ws);
    if (rc != ELSAA_OK) return rc;
    return elsaa_check_status(ws, stream);
}

extern "C" int elsaa_selftest_wait_timeout_noalloc(int limit_ms,
                                                   void *stream) {
    void *ws = nullptr;
    int rc = static_workspace(&ws);
    if (rc != ELSAA_OK) return rc;
    return elsaa_selftest_wait_timeout(ws, ELSAA_STATIC_WORKSPACE_BYTES,
                                       limit_ms, stream);
}
