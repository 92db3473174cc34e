// Per-head projections of the MoSA layer on CUDA cores (fp32 FFMA), used for
// fp32 storage and as the plain path for bf16:
//   F3  Q, K, V = X^s W^{Q,K,V}           (X^s = X[b, I, :], Sec. 2.2)
//   F5  Y[b, I, :] += diag(r^topk) A W^o  (scatter-sum over heads, Eq. mosa_mha)
//   B1  G = dY[I] W^o^T, dW^o = (diag(r) A)^T dY[I], and the row terms
//       dr = <A, G>, dA = r G, dlogit = dr r (1 - r), D = rowsum(dA o A)
//   B3  dX[b, I, :] += dQ W^Q^T + dK W^K^T + dV W^V^T + dlogit W^r[:,h]^T
//   B4  dW^{Q,K,V} = X^s^T d{Q,K,V},  dW^r[:,h] = X^s^T dlogit
// Rows of head h are m = b*k + i; gidx maps them to rows of X / Y / dY.
#include <cstdlib>

#include "launch.h"
#include "simt_gemm.cuh"

namespace mosa {
namespace {

template <class T>
struct QkvOp {
    using TS = typename InterOf<T>::type;
    static constexpr bool kAKFast = true, kBKFast = false;
    int M, N, K;  // B*k, 3*hp, d
    int hp;
    const T *X, *Wq, *Wk, *Wv;
    const int32_t *gidx;
    void *Q, *Kp, *V;
    __device__ float a(int g, int m, int c) const {
        return to_f32(X[(size_t)gidx[(size_t)g * M + m] * K + c]);
    }
    __device__ float b(int g, int c, int n) const {
        const int w = n / hp, p = n - w * hp;
        const T *W = w == 0 ? Wq : (w == 1 ? Wk : Wv);
        return to_f32(W[((size_t)g * K + c) * hp + p]);
    }
    __device__ void store(int g, int m, int n, float v) const {
        const int w = n / hp, p = n - w * hp;
        void *O = w == 0 ? Q : (w == 1 ? Kp : V);
        Inter<TS>::st(O, (size_t)g * M + m, hp, p, v);
    }
};

template <class T>
struct OutOp {
    using TS = typename InterOf<T>::type;
    static constexpr bool kAKFast = true, kBKFast = false;
    int M, N, K;  // B*k, d, hp
    const void *AR;
    const T *Wo;
    const int32_t *gidx;
    float *Y;
    __device__ float a(int g, int m, int p) const { return Inter<TS>::ld(AR, (size_t)g * M + m, K, p); }
    __device__ float b(int g, int p, int n) const { return to_f32(Wo[((size_t)g * K + p) * N + n]); }
    __device__ void store(int g, int m, int n, float v) const {
        atomicAdd(Y + (size_t)gidx[(size_t)g * M + m] * N + n, v);
    }
};

template <class T>
struct OutBwdGOp {
    static constexpr bool kAKFast = true, kBKFast = true;
    int M, N, K;  // B*k, hp, d
    const T *dY, *Wo;
    const int32_t *gidx;
    float *G;
    __device__ float a(int g, int m, int c) const {
        return to_f32(dY[(size_t)gidx[(size_t)g * M + m] * K + c]);
    }
    __device__ float b(int g, int c, int n) const { return to_f32(Wo[((size_t)g * N + n) * K + c]); }
    __device__ void store(int g, int m, int n, float v) const { G[((size_t)g * M + m) * N + n] = v; }
};

template <class T>
struct OutBwdWOp {
    using TS = typename InterOf<T>::type;
    static constexpr bool kAKFast = false, kBKFast = false;
    int M, N, K;  // hp, d, B*k
    const void *AR;
    const T *dY;
    const int32_t *gidx;
    float *dWo;
    __device__ float a(int g, int p, int m) const { return Inter<TS>::ld(AR, (size_t)g * K + m, M, p); }
    __device__ float b(int g, int m, int n) const {
        return to_f32(dY[(size_t)gidx[(size_t)g * K + m] * N + n]);
    }
    __device__ void store(int g, int p, int n, float v) const { dWo[((size_t)g * M + p) * N + n] = v; }
};

template <class T>
struct InBwdOp {
    using TS = typename InterOf<T>::type;
    static constexpr bool kAKFast = true, kBKFast = true;
    int M, N, K;  // B*k, d, 3*hp
    int hp, H;
    const void *dQKV;
    const T *Wq, *Wk, *Wv, *Wr;
    const float *dlogit;
    const int32_t *gidx;
    float *dX;
    __device__ float a(int g, int m, int kk) const { return Inter<TS>::ld(dQKV, (size_t)g * M + m, K, kk); }
    __device__ float b(int g, int kk, int n) const {
        const int w = kk / hp, p = kk - w * hp;
        const T *W = w == 0 ? Wq : (w == 1 ? Wk : Wv);
        return to_f32(W[((size_t)g * N + n) * hp + p]);
    }
    __device__ void store(int g, int m, int n, float v) const {
        const size_t row = (size_t)g * M + m;
        v = fmaf(dlogit[row], to_f32(Wr[(size_t)n * H + g]), v);
        atomicAdd(dX + (size_t)gidx[row] * N + n, v);
    }
};

// dW_{q,k,v} and, as one extra output column, dW_r.
template <class T>
struct WBwdOp {
    using TS = typename InterOf<T>::type;
    static constexpr bool kAKFast = false, kBKFast = false;
    int M, N, K;  // d, 3*hp + 1, B*k
    int hp, H;
    const T *X;
    const void *dQKV;
    const float *dlogit;
    const int32_t *gidx;
    float *dWq, *dWk, *dWv, *dWr;
    __device__ float a(int g, int c, int m) const {
        return to_f32(X[(size_t)gidx[(size_t)g * K + m] * M + c]);
    }
    __device__ float b(int g, int m, int n) const {
        const size_t row = (size_t)g * K + m;
        return n < 3 * hp ? Inter<TS>::ld(dQKV, row, 3 * hp, n) : dlogit[row];
    }
    __device__ void store(int g, int c, int n, float v) const {
        if (n == 3 * hp) {
            dWr[(size_t)c * H + g] = v;
            return;
        }
        const int w = n / hp, p = n - w * hp;
        float *O = w == 0 ? dWq : (w == 1 ? dWk : dWv);
        O[((size_t)g * M + c) * hp + p] = v;
    }
};

// One warp per selected row: dr = <A, G>, dA = r G (rounded to storage),
// D = rowsum(dA o A), dlogit = dr r (1 - r).
template <class TS>
__global__ void out_bwd_rows_kernel(const float *__restrict__ G, const float *__restrict__ A,
                                    const float *__restrict__ rsel, void *__restrict__ dA,
                                    float *__restrict__ Dd, float *__restrict__ dlogit,
                                    long long rows, int hp) {
    const long long row = (long long)blockIdx.x * (blockDim.x / 32) + threadIdx.x / 32;
    const int lane = threadIdx.x & 31;
    if (row >= rows) return;
    const float r = rsel[row];
    float dr = 0.f, dd = 0.f;
    for (int p = lane; p < hp; p += 32) {
        const float g = G[row * hp + p];
        const float a = A[row * hp + p];
        dr = fmaf(a, g, dr);
        const float da = r * g;
        Inter<TS>::st(dA, row, hp, p, da);
        dd = fmaf(da, a, dd);
    }
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) {
        dr += __shfl_xor_sync(0xffffffffu, dr, off);
        dd += __shfl_xor_sync(0xffffffffu, dd, off);
    }
    if (lane == 0) {
        Dd[row] = dd;
        dlogit[row] = dr * r * (1.f - r);
    }
}

// dW_r[c, h] = sum_m X[g(m), c] dlogit(m): one thread per column c of one
// head and one slice of the rows; slices are summed with atomics.
template <class T>
__global__ void dwr_kernel(const T *__restrict__ X, const int32_t *__restrict__ gidx,
                           const float *__restrict__ dlogit, float *__restrict__ dWr, int Mtok,
                           int d, int H, int rows_per_slice) {
    const int c = blockIdx.x * blockDim.x + threadIdx.x;
    const int h = blockIdx.y;
    const int m_begin = blockIdx.z * rows_per_slice;
    const int m_end = min(Mtok, m_begin + rows_per_slice);
    if (c >= d) return;
    float acc = 0.f;
    for (int m = m_begin; m < m_end; ++m) {
        const size_t row = (size_t)h * Mtok + m;
        acc = fmaf(to_f32(X[(size_t)gidx[row] * d + c]), dlogit[row], acc);
    }
    atomicAdd(dWr + (size_t)c * H + h, acc);
}

template <class T>
cudaError_t dwr_t(const Dims &dm, const void *X, const Saved &sv, float *dWr, cudaStream_t s) {
    cudaError_t e = cudaMemsetAsync(dWr, 0, sizeof(float) * (size_t)dm.d * dm.H, s);
    if (e != cudaSuccess) return e;
    const int Mtok = dm.B * dm.k;
    const int rows = 64;
    dim3 grid((dm.d + 255) / 256, dm.H, (Mtok + rows - 1) / rows);
    dwr_kernel<T><<<grid, 256, 0, s>>>((const T *)X, sv.gidx, sv.dlogit, dWr, Mtok, dm.d, dm.H,
                                       rows);
    note_launches(1);
    return cudaGetLastError();
}

template <class T>
cudaError_t qkv_t(const Dims &dm, const void *X, const void *Wq, const void *Wk, const void *Wv,
                  const Saved &sv, cudaStream_t s) {
    QkvOp<T> op{dm.B * dm.k, 3 * dm.hp, dm.d, dm.hp, (const T *)X, (const T *)Wq, (const T *)Wk,
                (const T *)Wv, sv.gidx, sv.Q, sv.K, sv.V};
    return launch_simt_gemm(op, dm.H, s);
}

template <class T>
cudaError_t out_t(const Dims &dm, const void *Wo, const Saved &sv, float *Y, cudaStream_t s) {
    if (!dm.accumulate) {
        cudaError_t e = cudaMemsetAsync(Y, 0, sizeof(float) * (size_t)dm.B * dm.T * dm.d, s);
        if (e != cudaSuccess) return e;
    }
    OutOp<T> op{dm.B * dm.k, dm.d, dm.hp, sv.AR, (const T *)Wo, sv.gidx, Y};
    return launch_simt_gemm(op, dm.H, s);
}

template <class T>
cudaError_t out_bwd_t(const Dims &dm, const void *Wo, const void *dY, const Saved &sv,
                      float *dWo, cudaStream_t s) {
    OutBwdGOp<T> g{dm.B * dm.k, dm.hp, dm.d, (const T *)dY, (const T *)Wo, sv.gidx, sv.G};
    cudaError_t e = launch_simt_gemm(g, dm.H, s);
    if (e != cudaSuccess) return e;
    const long long rows = dm.rows();
    const int warps = 8;
    out_bwd_rows_kernel<typename InterOf<T>::type>
        <<<(unsigned)((rows + warps - 1) / warps), warps * 32, 0, s>>>(
            sv.G, sv.A, sv.rsel, sv.dA, sv.Dd, sv.dlogit, rows, dm.hp);
    note_launches(1);
    if ((e = cudaGetLastError()) != cudaSuccess) return e;
    OutBwdWOp<T> w{dm.hp, dm.d, dm.B * dm.k, sv.AR, (const T *)dY, sv.gidx, dWo};
    return launch_simt_gemm(w, dm.H, s);
}

template <class T>
cudaError_t in_bwd_t(const Dims &dm, const void *Wq, const void *Wk, const void *Wv,
                     const void *Wr, const Saved &sv, float *dX, cudaStream_t s) {
    if (!dm.accumulate) {
        cudaError_t e = cudaMemsetAsync(dX, 0, sizeof(float) * (size_t)dm.B * dm.T * dm.d, s);
        if (e != cudaSuccess) return e;
    }
    InBwdOp<T> op{dm.B * dm.k, dm.d, 3 * dm.hp, dm.hp, dm.H, sv.dQKV, (const T *)Wq,
                  (const T *)Wk, (const T *)Wv, (const T *)Wr, sv.dlogit, sv.gidx, dX};
    return launch_simt_gemm(op, dm.H, s);
}

template <class T>
cudaError_t w_bwd_t(const Dims &dm, const void *X, const Saved &sv, float *dWq, float *dWk,
                    float *dWv, float *dWr, cudaStream_t s) {
    WBwdOp<T> op{dm.d, 3 * dm.hp + 1, dm.B * dm.k, dm.hp, dm.H, (const T *)X,
                 sv.dQKV, sv.dlogit, sv.gidx, dWq, dWk, dWv, dWr};
    return launch_simt_gemm(op, dm.H, s);
}

}  // namespace

bool use_tc(const Dims &dm) {
    const char *f = std::getenv("MOSA_FORCE_SIMT");
    if (f != nullptr && f[0] != '\0' && f[0] != '0') return false;
    return tc_supported(dm);
}

bool use_fused_forward(const Dims &dm) {
    const char *f = std::getenv("MOSA_FUSED_FWD");
    if (f != nullptr && f[0] == '0') return false;
    return use_tc(dm) && tc_fused_forward_supported(dm);
}

cudaError_t launch_qkv(const Dims &dm, const void *X, const void *Wq, const void *Wk,
                       const void *Wv, const Saved &sv, cudaStream_t s) {
    if (use_tc(dm)) return tc_qkv(dm, X, Wq, Wk, Wv, sv, s);
    return dm.bf16 ? qkv_t<bf16>(dm, X, Wq, Wk, Wv, sv, s) : qkv_t<float>(dm, X, Wq, Wk, Wv, sv, s);
}

cudaError_t launch_out(const Dims &dm, const void *Wo, const Saved &sv, float *Y, cudaStream_t s) {
    if (use_tc(dm)) return tc_out(dm, Wo, sv, Y, s, !dm.accumulate);
    return dm.bf16 ? out_t<bf16>(dm, Wo, sv, Y, s) : out_t<float>(dm, Wo, sv, Y, s);
}

cudaError_t launch_out_bwd(const Dims &dm, const void *Wo, const void *dY, const Saved &sv,
                           float *dWo, cudaStream_t s) {
    if (use_tc(dm)) {
        cudaError_t e = tc_out_bwd_g(dm, Wo, dY, sv, s);
        return e != cudaSuccess ? e : tc_out_bwd_w(dm, dY, sv, dWo, s);
    }
    return dm.bf16 ? out_bwd_t<bf16>(dm, Wo, dY, sv, dWo, s) : out_bwd_t<float>(dm, Wo, dY, sv, dWo, s);
}

cudaError_t launch_in_bwd(const Dims &dm, const void *Wq, const void *Wk, const void *Wv,
                          const void *Wr, const Saved &sv, float *dX, cudaStream_t s) {
    if (use_tc(dm)) {
        cudaError_t e = tc_transpose_wr(dm, Wr, sv, s);
        return e != cudaSuccess ? e : tc_in_bwd(dm, Wq, Wk, Wv, Wr, sv, dX, s, !dm.accumulate);
    }
    return dm.bf16 ? in_bwd_t<bf16>(dm, Wq, Wk, Wv, Wr, sv, dX, s)
                   : in_bwd_t<float>(dm, Wq, Wk, Wv, Wr, sv, dX, s);
}

cudaError_t launch_w_bwd(const Dims &dm, const void *X, const Saved &sv, float *dWq, float *dWk,
                         float *dWv, float *dWr, cudaStream_t s) {
    if (use_tc(dm)) return tc_w_bwd(dm, X, sv, dWq, dWk, dWv, dWr, s);
    return dm.bf16 ? w_bwd_t<bf16>(dm, X, sv, dWq, dWk, dWv, dWr, s)
                   : w_bwd_t<float>(dm, X, sv, dWq, dWk, dWv, dWr, s);
}

}  // namespace mosa
