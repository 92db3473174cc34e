// Routing (router scores + TopK selection) for callers that cannot allocate
// device memory.
//
// mosa_forward keeps the [B,H,T] router scores in the caller's workspace.
// Some callers have no way to provide one: code running inside a host
// application that owns the whole device heap and hands out no buffers after
// start-up, plug-ins whose interface only passes input and output tensors,
// or loops that must never trigger cudaMalloc's implicit device-wide
// synchronisation.  For them mosa_route_noalloc keeps the scores in a fixed
// array compiled into this library instead.
#include "../../include/mosa.h"
#include "launch.h"

namespace mosa {
namespace {

// Largest B*H*T the array holds: 2^20 fp32 scores, 4 MiB per GPU that loads
// the library, resident until the process exits.
constexpr size_t kRouteScratchScores = size_t(1) << 20;

__device__ __align__(256) float g_route_scores[kRouteScratchScores];

// Status word for the router's bounded waits (there is no workspace to hold
// one).  Nothing reads it back: a wait that runs out (a GPU that stopped
// making progress for 2 s) leaves that call's I and r_sel undefined.
__device__ __align__(256) uint32_t g_route_status;

// Device addresses of the two arrays on the current device.  They are looked
// up on every call (cheap once the library's device code is loaded) rather
// than cached: a device reset reloads the module, and a cached address could
// then point at freed memory.  The host-side symbols are only stand-ins and
// must never reach a kernel.
cudaError_t scratch_addresses(float **scores, uint32_t **status) {
    void *p = nullptr;
    cudaError_t e = cudaGetSymbolAddress(&p, g_route_scores);
    if (e != cudaSuccess) return e;
    *scores = static_cast<float *>(p);
    e = cudaGetSymbolAddress(&p, g_route_status);
    if (e != cudaSuccess) return e;
    *status = static_cast<uint32_t *>(p);
    return cudaSuccess;
}

}  // namespace
}  // namespace mosa

using namespace mosa;

extern "C" mosa_status mosa_route_noalloc(const mosa_shape *shape, const void *X,
                                          const void *W_r, int32_t *I, float *r_sel,
                                          void *stream) {
    if (mosa_workspace_bytes(shape) == 0) {
        // invalid or unsupported shape: report which
        if (shape == nullptr || shape->B <= 0 || shape->T <= 0 || shape->d <= 0 ||
            shape->H <= 0 || shape->hp <= 0 || shape->k <= 0 || shape->k > shape->T ||
            (shape->dtype != MOSA_F32 && shape->dtype != MOSA_BF16) ||
            (shape->first_token != 0 && shape->first_token != 1) ||
            (shape->rope != 0 && shape->rope != 1))
            return MOSA_ERR_INVALID_ARG;
        return MOSA_ERR_UNSUPPORTED;
    }
    if (X == nullptr || W_r == nullptr || I == nullptr || r_sel == nullptr)
        return MOSA_ERR_INVALID_ARG;
    if ((size_t)shape->B * shape->H * shape->T > kRouteScratchScores) return MOSA_ERR_UNSUPPORTED;
    float *scores = nullptr;
    uint32_t *status = nullptr;
    if (scratch_addresses(&scores, &status) != cudaSuccess) return MOSA_ERR_CUDA;
    const Dims dm{shape->B, shape->T, shape->d, shape->H, shape->hp, shape->k,
                  shape->dtype == MOSA_BF16, shape->first_token != 0, shape->rope != 0};
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    // Every score the selection reads is written by the router first, so the
    // array needs no clearing between calls.  The router is chosen as in
    // mosa_forward (tensor cores for bf16 with H % 8 == 0), so both entry
    // points compute the same scores bit for bit.
    if (launch_router_auto(dm, X, W_r, scores, status, s) != cudaSuccess) return MOSA_ERR_CUDA;
    if (launch_select(dm.B * dm.H, dm.T, dm.k, scores, I, r_sel, 0, 1, nullptr, nullptr, s,
                      dm.first_token) !=
        cudaSuccess)
        return MOSA_ERR_CUDA;
    return MOSA_OK;
}
