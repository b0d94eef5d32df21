// elsaa_forward_noalloc: the forward pass with scratch taken from a fixed
// array in the library's device image, for callers that cannot allocate
// device memory (see include/elsaa.h for the contract).
#include <mutex>

#include "internal.h"

namespace {

// The scratch array. In host code this name is only a host-side handle for
// the device symbol, never a device address: its device address is looked
// up with cudaGetSymbolAddress below, once per device.
static __device__ __align__(256) unsigned char
    g_static_workspace[ELSAA_STATIC_WORKSPACE_BYTES];

constexpr int kMaxDevices = 64;
void *g_static_ptr[kMaxDevices] = {};
std::mutex g_static_mu;

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
    int dev = -1;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess)
        return elsaa::set_last_error(ELSAA_ERR_CUDA, "cudaGetDevice: %s",
                                     cudaGetErrorString(e));
    if (dev < 0 || dev >= kMaxDevices)
        return elsaa::set_last_error(ELSAA_ERR_UNSUPPORTED,
                                     "device ordinal %d above %d", dev,
                                     kMaxDevices - 1);
    void *ws = nullptr;
    {
        std::lock_guard<std::mutex> lk(g_static_mu);
        if (!g_static_ptr[dev]) {
            // set-up, once per device, with that device current
            void *p = nullptr;
            e = cudaGetSymbolAddress(&p, g_static_workspace);
            if (e != cudaSuccess || !p)
                return elsaa::set_last_error(
                    ELSAA_ERR_CUDA, "cudaGetSymbolAddress: %s",
                    cudaGetErrorString(e));
            g_static_ptr[dev] = p;
        }
        ws = g_static_ptr[dev];
    }
    return elsaa_forward(params, q, k, v, w_sort, w_race, lambda_tok, gates,
                         o, log_d_sparse, d_lr, m_sparse, perm_q, perm_k, ws,
                         ELSAA_STATIC_WORKSPACE_BYTES, stream);
}
