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
    kStatusRange = 4u,     // an fp16 intermediate of the k > 128 attention overflowed
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

// Intermediates (Q, K, V, diag(r) A, dA, dQ|dK|dV) are kept at about fp32
// precision whatever the input dtype: fp32 arrays for fp32 inputs, and for
// bf16 inputs a pair (hi, lo) of bf16 values with v ~= hi + lo (hi = bf16(v),
// lo = bf16(v - hi)), stored as planar halves of each row: [hi x cols | lo x
// cols].  A tensor-core product with such an operand is two bf16 MMAs into
// one fp32 accumulator.  Both forms take 4 bytes per element.
struct SplitBF16 {};

template <class TS>
struct Inter;

template <>
struct Inter<float> {
    static __device__ __forceinline__ float ld(const void *p, size_t row, int cols, int c) {
        return static_cast<const float *>(p)[row * cols + c];
    }
    static __device__ __forceinline__ void st(void *p, size_t row, int cols, int c, float v) {
        static_cast<float *>(p)[row * cols + c] = v;
    }
};

template <>
struct Inter<SplitBF16> {
    static __device__ __forceinline__ float ld(const void *p, size_t row, int cols, int c) {
        const bf16 *q = static_cast<const bf16 *>(p) + row * 2 * cols;
        return __bfloat162float(q[c]) + __bfloat162float(q[cols + c]);
    }
    static __device__ __forceinline__ void st(void *p, size_t row, int cols, int c, float v) {
        bf16 *q = static_cast<bf16 *>(p) + row * 2 * cols;
        const bf16 hi = __float2bfloat16_rn(v);
        q[c] = hi;
        q[cols + c] = __float2bfloat16_rn(v - __bfloat162float(hi));
    }
};

// Intermediate storage for an input dtype.
template <class TI>
struct InterOf {
    using type = float;
};
template <>
struct InterOf<bf16> {
    using type = SplitBF16;
};

// Internal views of the workspace.  Per-head state is stored head-major,
// [H][B*k][...], so that each head's B*k selected rows form one contiguous
// matrix (row m = b*k + i).
struct Saved {
    uint32_t *status;   // device status word
    float *r_full;      // [B,H,T]   router scores (when the caller gives none)
    int32_t *gidx;      // [H,B*k]   b*T + I[b,h,i]: row of X / Y / dY to gather or scatter
    float *rsel;        // [H,B*k]   r^topk in the same order
    void *Q, *K, *V;    // [H,B*k,hp] intermediate (fp32 or bf16 hi/lo pair)
    float *A;           // [H,B*k,hp] attention output, fp32
    void *AR;           // [H,B*k,hp] diag(r^topk) A, intermediate
    float *lse;         // [H,B*k]   log-sum-exp of the scaled, masked scores
    void *dA;           // [H,B*k,hp] gradient of A, intermediate
    float *dlogit;      // [H,B*k]   gradient of the router logit
    float *Dd;          // [H,B*k]   rowsum(dA o A)
    void *dQKV;         // [H,B*k,3hp] dQ | dK | dV, intermediate (tensor-core path:
                        // [H,B*k,512] bf16 pair dQ|dK|dV|dlogit,0.. hi then lo)
    float *G;           // [H,B*k,hp] dY[I] W_o^T (fp32, CUDA-core path); on the
                        // tensor-core path with k > 128 the fp32 dQ accumulator
    float *WrT;         // [H,d] fp32 transpose of W_r (tensor-core dX epilogue)
    void *Wr64;         // [d, H rounded up to 64] bf16 W_r with zero columns past H
                        // (tensor-core router, H % 64 != 0)
    // fp16 dQ|dK|dV rows (tensor cores: k > 128, and k <= 128 where the
    // weights' copy is small, dqkv_f16): dQKV is [H,B*k,256] fp16
    // (dQ | dK | dV | dlogit, 0..), and the backward reads X and W_q|W_k|W_v
    // through fp16 copies so that every product with dQKV is one MMA
    void *X16;          // [B*T,d] fp16 copy of X
    void *W16;          // [3][H,d,hp] fp16 copies of W_q, W_k, W_v, then [H,hp,d] of W_o
    void *AR16;         // [H,B*k,hp] fp16 diag(r^topk) A (the output product's operand)
    unsigned long long *spans;   // [16][2] kernel spans of the timed stages (measurement)
    int32_t *pos;       // [H,B*T] row b*k + i of head h holding token (b, t), or -1
                        // (token-major output and input-gradient products, k > 128)
};

// Rotary position encoding (Sec. 2.2): pair p of the first h'/2 dimensions of
// a query or key row at original position t turns by t * theta_p, theta_p =
// 10000^(-2p / (h'/2)).  phi[p] holds theta_p / (2 pi) in turns per position
// as a 64-bit fixed-point fraction, so t * phi[p] taken mod 2^64 is the angle's
// fraction of a turn, exact up to phi's rounding (about 1e-12 rad at t =
// 65535), for any t: no large angle ever reaches a floating-point sin or cos.
constexpr int kRopeMaxPairs = 32;   // h' <= 128
struct RopeTable {
    uint64_t phi[kRopeMaxPairs];
    int npairs;   // h' / 4
    int T;        // positions are gidx mod T
};

// (x0, x1) turned by dir * t * theta (dir = +1 forward, -1 for gradients).
// The top 24 bits of the turn fraction, read as signed, give the angle in
// [-pi, pi), where the hardware sine and cosine are accurate to about 4e-7.
__device__ __forceinline__ void rope_turn(float &x0, float &x1, uint64_t phi, int t, float dir) {
    const uint64_t turns = phi * (uint64_t)(uint32_t)t;               // mod one turn
    const int32_t q = (int32_t)(uint32_t)(turns >> 32) >> 8;          // [-2^23, 2^23)
    const float ang = (float)q * (6.2831853071795865f / 16777216.f);  // [-pi, pi)
    float sn, cs;
    __sincosf(ang, &sn, &cs);
    sn *= dir;
    const float y0 = x0 * cs - x1 * sn, y1 = x0 * sn + x1 * cs;
    x0 = y0;
    x1 = y1;
}

// Kernel spans (measurement only): a stage's kernels record the earliest
// start and the latest end of their CTAs (%globaltimer, ns) into a slot
// [start, end] of the workspace, when that stage is being timed (sp != null).
__device__ __forceinline__ unsigned long long span_clock() {
    unsigned long long t;
    asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
    return t;
}
__device__ __forceinline__ void span_begin(unsigned long long *sp) {
    if (sp != nullptr && threadIdx.x == 0) atomicMin(sp, span_clock());
}
// Call after the CTA's last barrier (all its work done).
__device__ __forceinline__ void span_end(unsigned long long *sp) {
    if (sp != nullptr && threadIdx.x == 0) atomicMax(sp + 1, span_clock());
}

struct Dims {
    int B, T, d, H, hp, k;
    bool bf16;
    bool first_token;   // token 0 always kept, k-1 more by score (Sec. 3.2)
    bool rope;          // rotary position encoding of Q and K (Sec. 2.2)
    bool accumulate;    // Y (forward) and dX (backward) are added into, not overwritten
    long long rows() const { return (long long)H * B * k; }
    size_t esize() const { return bf16 ? 2 : 4; }
};

}  // namespace mosa
