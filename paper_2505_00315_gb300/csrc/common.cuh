// Device-side helpers shared by the libmosa kernels: dtype conversion, the
// workspace status word and the internal layout of saved per-head state.
#pragma once

#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include <cstddef>
#include <cstdint>

namespace mosa {

// Bits of the device status word kept at the start of the workspace.
enum : uint32_t {
    kStatusBadIndex = 1u,  // caller-supplied indices out of range or not ascending
    kStatusTimeout = 2u,   // a bounded spin-wait gave up
};

using bf16 = __nv_bfloat16;

__device__ __forceinline__ float to_f32(float x) { return x; }
__device__ __forceinline__ float to_f32(bf16 x) { return __bfloat162float(x); }

template <class T>
__device__ __forceinline__ T from_f32(float x);
template <>
__device__ __forceinline__ float from_f32<float>(float x) { return x; }
template <>
__device__ __forceinline__ bf16 from_f32<bf16>(float x) { return __float2bfloat16_rn(x); }

// Internal views of the workspace.  Per-head state is stored head-major,
// [H][B*k][...], so that each head's B*k selected rows form one contiguous
// matrix (row m = b*k + i).
struct Saved {
    uint32_t *status;   // device status word
    float *r_full;      // [B,H,T]   router scores (when the caller gives none)
    int32_t *gidx;      // [H,B*k]   b*T + I[b,h,i]: row of X / Y / dY to gather or scatter
    float *rsel;        // [H,B*k]   r^topk in the same order
    void *Q, *K, *V;    // [H,B*k,hp] storage dtype
    void *A;            // [H,B*k,hp] attention output
    void *AR;           // [H,B*k,hp] diag(r^topk) A
    float *lse;         // [H,B*k]   log-sum-exp of the scaled, masked scores
    void *dA;           // [H,B*k,hp] gradient of A
    float *dlogit;      // [H,B*k]   gradient of the router logit
    float *Dd;          // [H,B*k]   rowsum(dA o A)
    void *dQKV;         // [H,B*k,3hp] dQ | dK | dV
    float *G;           // [H,B*k,hp] dY[I] W_o^T (fp32)
};

struct Dims {
    int B, T, d, H, hp, k;
    bool bf16;
    long long rows() const { return (long long)H * B * k; }
    size_t esize() const { return bf16 ? 2 : 4; }
};

}  // namespace mosa
