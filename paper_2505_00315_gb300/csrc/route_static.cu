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
#include <mutex>

#include "../../include/mosa.h"
#include "launch.h"

namespace mosa {
namespace {

// Largest B*H*T the array holds: 2^20 fp32 scores, 4 MiB per GPU that loads
// the library, resident until the process exits.
constexpr size_t kRouteScratchScores = size_t(1) << 20;

__device__ __align__(256) float g_route_scores[kRouteScratchScores];

constexpr int kMaxDevices = 64;
std::mutex g_mu;
float *g_scores_on[kMaxDevices] = {};

// Device address of g_route_scores on the current device, looked up once per
// device (the host-side symbol is only a stand-in and must not reach a kernel).
cudaError_t scores_address(float **out) {
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    if (dev < 0 || dev >= kMaxDevices) return cudaErrorInvalidDevice;
    std::lock_guard<std::mutex> lk(g_mu);
    if (g_scores_on[dev] == nullptr) {
        void *p = nullptr;
        e = cudaGetSymbolAddress(&p, g_route_scores);
        if (e != cudaSuccess) return e;
        g_scores_on[dev] = static_cast<float *>(p);
    }
    *out = g_scores_on[dev];
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
    if (scores_address(&scores) != cudaSuccess) return MOSA_ERR_CUDA;
    const Dims dm{shape->B, shape->T, shape->d, shape->H, shape->hp, shape->k,
                  shape->dtype == MOSA_BF16, shape->first_token != 0, shape->rope != 0};
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    // Every score the selection reads is written by the router first, so the
    // array needs no clearing between calls.
    if (launch_router(dm, X, W_r, scores, s) != cudaSuccess) return MOSA_ERR_CUDA;
    if (launch_select(dm.B * dm.H, dm.T, dm.k, scores, I, r_sel, 0, 1, nullptr, nullptr, s,
                      dm.first_token) !=
        cudaSuccess)
        return MOSA_ERR_CUDA;
    return MOSA_OK;
}
