// Index-masked causal attention over the k selected tokens of each head
// (Sec. 2.1 Eq. attention, Sec. 2.2 mask M_ij = 0 iff I_i >= I_j) on CUDA
// cores, fp32 arithmetic.  I is strictly ascending, so I_i >= I_j is j <= i.
//
// Forward (F4): one thread per query row, online softmax over key tiles kept
// in shared memory; writes A, diag(r^topk) A and the row log-sum-exp.
// Backward (B2): P is recomputed from the saved log-sum-exp;
//   dP = dA V^T, dS = P o (dP - D), dQ = dS K / sqrt(h'), dK = dS^T Q / sqrt(h'),
//   dV = P^T dA, with D = rowsum(dA o A),
// one thread per query row (dQ) or per key row (dK, dV).
#include <cfloat>

#include "launch.h"
#include "profile.h"

namespace mosa {
namespace {

constexpr int kRowsPerBlock = 64;
constexpr int kTile = 32;

template <class TS, int HP>
__global__ void __launch_bounds__(kRowsPerBlock)
attn_fwd_simt_kernel(const void *__restrict__ Q, const void *__restrict__ K,
                     const void *__restrict__ V, const float *__restrict__ rsel,
                     float *__restrict__ A, void *__restrict__ AR, float *__restrict__ lse, int k,
                     float scale) {
    __shared__ float Ks[kTile][HP], Vs[kTile][HP];
    const size_t base = (size_t)blockIdx.y * k;
    const int i = blockIdx.x * kRowsPerBlock + threadIdx.x;
    float q[HP], o[HP];
#pragma unroll
    for (int p = 0; p < HP; ++p) {
        q[p] = i < k ? Inter<TS>::ld(Q, base + i, HP, p) * scale : 0.f;
        o[p] = 0.f;
    }
    float m = -FLT_MAX, l = 0.f;
    const int last = min(k, (int)(blockIdx.x + 1) * kRowsPerBlock) - 1;
    for (int j0 = 0; j0 <= last; j0 += kTile) {
        __syncthreads();
        for (int e = threadIdx.x; e < kTile * HP; e += kRowsPerBlock) {
            const int jj = e / HP, p = e % HP, j = j0 + jj;
            Ks[jj][p] = j < k ? Inter<TS>::ld(K, base + j, HP, p) : 0.f;
            Vs[jj][p] = j < k ? Inter<TS>::ld(V, base + j, HP, p) : 0.f;
        }
        __syncthreads();
        if (i < k) {
            const int jn = min(kTile, i - j0 + 1);
            for (int jj = 0; jj < jn; ++jj) {
                float s = 0.f;
#pragma unroll
                for (int p = 0; p < HP; ++p) s = fmaf(q[p], Ks[jj][p], s);
                if (s > m) {
                    const float corr = expf(m - s);
                    l *= corr;
#pragma unroll
                    for (int p = 0; p < HP; ++p) o[p] *= corr;
                    m = s;
                }
                const float pr = expf(s - m);
                l += pr;
#pragma unroll
                for (int p = 0; p < HP; ++p) o[p] = fmaf(pr, Vs[jj][p], o[p]);
            }
        }
    }
    if (i < k) {
        const float inv = 1.f / l, r = rsel[base + i];
#pragma unroll
        for (int p = 0; p < HP; ++p) {
            const float a = o[p] * inv;
            A[(base + i) * HP + p] = a;
            Inter<TS>::st(AR, base + i, HP, p, r * a);
        }
        lse[base + i] = m + logf(l);
    }
}

// dQ: one thread per query row i, keys j <= i.
template <class TS, int HP>
__global__ void __launch_bounds__(kRowsPerBlock)
attn_bwd_dq_simt_kernel(const void *__restrict__ Q, const void *__restrict__ K,
                        const void *__restrict__ V, const void *__restrict__ dA,
                        const float *__restrict__ lse, const float *__restrict__ Dd,
                        void *__restrict__ dQKV, int k, float scale) {
    __shared__ float Ks[kTile][HP], Vs[kTile][HP];
    const size_t base = (size_t)blockIdx.y * k;
    const int i = blockIdx.x * kRowsPerBlock + threadIdx.x;
    float q[HP], da[HP], dq[HP];
#pragma unroll
    for (int p = 0; p < HP; ++p) {
        q[p] = i < k ? Inter<TS>::ld(Q, base + i, HP, p) * scale : 0.f;
        da[p] = i < k ? Inter<TS>::ld(dA, base + i, HP, p) : 0.f;
        dq[p] = 0.f;
    }
    const float L = i < k ? lse[base + i] : 0.f, D = i < k ? Dd[base + i] : 0.f;
    const int last = min(k, (int)(blockIdx.x + 1) * kRowsPerBlock) - 1;
    for (int j0 = 0; j0 <= last; j0 += kTile) {
        __syncthreads();
        for (int e = threadIdx.x; e < kTile * HP; e += kRowsPerBlock) {
            const int jj = e / HP, p = e % HP, j = j0 + jj;
            Ks[jj][p] = j < k ? Inter<TS>::ld(K, base + j, HP, p) : 0.f;
            Vs[jj][p] = j < k ? Inter<TS>::ld(V, base + j, HP, p) : 0.f;
        }
        __syncthreads();
        if (i < k) {
            const int jn = min(kTile, i - j0 + 1);
            for (int jj = 0; jj < jn; ++jj) {
                float s = 0.f, dp = 0.f;
#pragma unroll
                for (int p = 0; p < HP; ++p) {
                    s = fmaf(q[p], Ks[jj][p], s);
                    dp = fmaf(da[p], Vs[jj][p], dp);
                }
                const float ds = expf(s - L) * (dp - D);
#pragma unroll
                for (int p = 0; p < HP; ++p) dq[p] = fmaf(ds, Ks[jj][p], dq[p]);
            }
        }
    }
    if (i < k) {
#pragma unroll
        for (int p = 0; p < HP; ++p) Inter<TS>::st(dQKV, base + i, 3 * HP, p, dq[p] * scale);
    }
}

// dK and dV: one thread per key row j, queries i >= j.
template <class TS, int HP, bool kDK>
__global__ void __launch_bounds__(kRowsPerBlock)
attn_bwd_dkv_simt_kernel(const void *__restrict__ Q, const void *__restrict__ K,
                         const void *__restrict__ V, const void *__restrict__ dA,
                         const float *__restrict__ lse, const float *__restrict__ Dd,
                         void *__restrict__ dQKV, int k, float scale) {
    __shared__ float Qs[kTile][HP], dAs[kTile][HP], Ls[kTile], Ds[kTile];
    const size_t base = (size_t)blockIdx.y * k;
    const int j = blockIdx.x * kRowsPerBlock + threadIdx.x;
    float kr[HP], vr[HP], acc[HP];
#pragma unroll
    for (int p = 0; p < HP; ++p) {
        kr[p] = j < k ? Inter<TS>::ld(K, base + j, HP, p) * scale : 0.f;
        vr[p] = (kDK && j < k) ? Inter<TS>::ld(V, base + j, HP, p) : 0.f;
        acc[p] = 0.f;
    }
    for (int i0 = blockIdx.x * kRowsPerBlock; i0 < k; i0 += kTile) {
        __syncthreads();
        for (int e = threadIdx.x; e < kTile * HP; e += kRowsPerBlock) {
            const int ii = e / HP, p = e % HP, i = i0 + ii;
            Qs[ii][p] = i < k ? Inter<TS>::ld(Q, base + i, HP, p) : 0.f;
            dAs[ii][p] = i < k ? Inter<TS>::ld(dA, base + i, HP, p) : 0.f;
        }
        for (int ii = threadIdx.x; ii < kTile; ii += kRowsPerBlock) {
            const int i = i0 + ii;
            Ls[ii] = i < k ? lse[base + i] : 0.f;
            Ds[ii] = i < k ? Dd[base + i] : 0.f;
        }
        __syncthreads();
        if (j < k) {
            const int iend = min(kTile, k - i0);
            for (int ii = max(0, j - i0); ii < iend; ++ii) {
                float s = 0.f, dp = 0.f;
#pragma unroll
                for (int p = 0; p < HP; ++p) {
                    s = fmaf(Qs[ii][p], kr[p], s);
                    if (kDK) dp = fmaf(dAs[ii][p], vr[p], dp);
                }
                const float pr = expf(s - Ls[ii]);
                if (kDK) {
                    const float ds = pr * (dp - Ds[ii]);
#pragma unroll
                    for (int p = 0; p < HP; ++p) acc[p] = fmaf(ds, Qs[ii][p], acc[p]);
                } else {
#pragma unroll
                    for (int p = 0; p < HP; ++p) acc[p] = fmaf(pr, dAs[ii][p], acc[p]);
                }
            }
        }
    }
    if (j < k) {
        const int col = kDK ? HP : 2 * HP;
        const float f = kDK ? scale : 1.f;
#pragma unroll
        for (int p = 0; p < HP; ++p) Inter<TS>::st(dQKV, base + j, 3 * HP, col + p, acc[p] * f);
    }
}

template <class TS, int HP>
cudaError_t attn_fwd_t(const Dims &dm, const Saved &sv, cudaStream_t s) {
    dim3 grid((dm.k + kRowsPerBlock - 1) / kRowsPerBlock, dm.H * dm.B);
    const float scale = 1.f / sqrtf((float)HP);
    attn_fwd_simt_kernel<TS, HP><<<grid, kRowsPerBlock, 0, s>>>(sv.Q, sv.K, sv.V, sv.rsel, sv.A,
                                                               sv.AR, sv.lse, dm.k, scale);
    note_launches(1);
    return cudaGetLastError();
}

template <class TS, int HP>
cudaError_t attn_bwd_t(const Dims &dm, const Saved &sv, cudaStream_t s) {
    dim3 grid((dm.k + kRowsPerBlock - 1) / kRowsPerBlock, dm.H * dm.B);
    const float scale = 1.f / sqrtf((float)HP);
    attn_bwd_dq_simt_kernel<TS, HP><<<grid, kRowsPerBlock, 0, s>>>(
        sv.Q, sv.K, sv.V, sv.dA, sv.lse, sv.Dd, sv.dQKV, dm.k, scale);
    attn_bwd_dkv_simt_kernel<TS, HP, true><<<grid, kRowsPerBlock, 0, s>>>(
        sv.Q, sv.K, sv.V, sv.dA, sv.lse, sv.Dd, sv.dQKV, dm.k, scale);
    attn_bwd_dkv_simt_kernel<TS, HP, false><<<grid, kRowsPerBlock, 0, s>>>(
        sv.Q, sv.K, sv.V, sv.dA, sv.lse, sv.Dd, sv.dQKV, dm.k, scale);
    note_launches(3);
    return cudaGetLastError();
}

template <class TS>
cudaError_t attn_fwd_dispatch(const Dims &dm, const Saved &sv, cudaStream_t s) {
    switch (dm.hp) {
        case 16: return attn_fwd_t<TS, 16>(dm, sv, s);
        case 32: return attn_fwd_t<TS, 32>(dm, sv, s);
        case 64: return attn_fwd_t<TS, 64>(dm, sv, s);
        case 128: return attn_fwd_t<TS, 128>(dm, sv, s);
        default: return cudaErrorInvalidValue;
    }
}

template <class TS>
cudaError_t attn_bwd_dispatch(const Dims &dm, const Saved &sv, cudaStream_t s) {
    switch (dm.hp) {
        case 16: return attn_bwd_t<TS, 16>(dm, sv, s);
        case 32: return attn_bwd_t<TS, 32>(dm, sv, s);
        case 64: return attn_bwd_t<TS, 64>(dm, sv, s);
        case 128: return attn_bwd_t<TS, 128>(dm, sv, s);
        default: return cudaErrorInvalidValue;
    }
}

}  // namespace

cudaError_t launch_attn_fwd(const Dims &dm, const Saved &sv, cudaStream_t s) {
    if (use_tc(dm)) return tc_attn_fwd(dm, sv, s);
    return dm.bf16 ? attn_fwd_dispatch<SplitBF16>(dm, sv, s) : attn_fwd_dispatch<float>(dm, sv, s);
}

cudaError_t launch_attn_bwd(const Dims &dm, const Saved &sv, cudaStream_t s, float *zero_out) {
    if (use_tc(dm)) return tc_attn_bwd(dm, sv, s, zero_out);
    return dm.bf16 ? attn_bwd_dispatch<SplitBF16>(dm, sv, s) : attn_bwd_dispatch<float>(dm, sv, s);
}

}  // namespace mosa
