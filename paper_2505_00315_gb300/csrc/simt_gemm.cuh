// Grouped SIMT (CUDA-core, fp32 FFMA) matrix product with caller-defined
// operand addressing.  It serves the fp32 storage path, where the tolerance
// rules out tensor-core TF32, and is the plain reference path for bf16 too.
//
// For every group g (blockIdx.z) it computes C[g](m,n) = sum_kk A(g,m,kk) B(g,kk,n)
// for 0 <= m < op.M, 0 <= n < op.N, 0 <= kk < op.K, reading elements through
// op.a(g,m,kk) / op.b(g,kk,n) and handing each result to op.store(g,m,n,acc).
// The functors carry the gathers (rows chosen by a head), transposes and
// scatter-adds of the MoSA steps.
#pragma once

#include "common.cuh"
#include "profile.h"

namespace mosa {

constexpr int kSimtBM = 64, kSimtBN = 64, kSimtBK = 16, kSimtThreads = 256;

template <class Op>
__global__ void __launch_bounds__(kSimtThreads) simt_gemm_kernel(Op op) {
    __shared__ float As[kSimtBK][kSimtBM + 4];
    __shared__ float Bs[kSimtBK][kSimtBN + 4];
    const int g = blockIdx.z;
    const int m0 = blockIdx.y * kSimtBM, n0 = blockIdx.x * kSimtBN;
    const int tid = threadIdx.x;
    const int tm = (tid / 16) * 4, tn = (tid % 16) * 4;
    float acc[4][4];
#pragma unroll
    for (int i = 0; i < 4; ++i)
#pragma unroll
        for (int j = 0; j < 4; ++j) acc[i][j] = 0.f;

    for (int k0 = 0; k0 < op.K; k0 += kSimtBK) {
        for (int e = tid; e < kSimtBM * kSimtBK; e += kSimtThreads) {
            const int mm = Op::kAKFast ? e / kSimtBK : e % kSimtBM;
            const int kk = Op::kAKFast ? e % kSimtBK : e / kSimtBM;
            const int m = m0 + mm, kx = k0 + kk;
            As[kk][mm] = (m < op.M && kx < op.K) ? op.a(g, m, kx) : 0.f;
        }
        for (int e = tid; e < kSimtBK * kSimtBN; e += kSimtThreads) {
            const int nn = Op::kBKFast ? e / kSimtBK : e % kSimtBN;
            const int kk = Op::kBKFast ? e % kSimtBK : e / kSimtBN;
            const int n = n0 + nn, kx = k0 + kk;
            Bs[kk][nn] = (n < op.N && kx < op.K) ? op.b(g, kx, n) : 0.f;
        }
        __syncthreads();
#pragma unroll
        for (int kk = 0; kk < kSimtBK; ++kk) {
            float a[4], b[4];
#pragma unroll
            for (int i = 0; i < 4; ++i) a[i] = As[kk][tm + i];
#pragma unroll
            for (int j = 0; j < 4; ++j) b[j] = Bs[kk][tn + j];
#pragma unroll
            for (int i = 0; i < 4; ++i)
#pragma unroll
                for (int j = 0; j < 4; ++j) acc[i][j] = fmaf(a[i], b[j], acc[i][j]);
        }
        __syncthreads();
    }
#pragma unroll
    for (int i = 0; i < 4; ++i)
#pragma unroll
        for (int j = 0; j < 4; ++j) {
            const int m = m0 + tm + i, n = n0 + tn + j;
            if (m < op.M && n < op.N) op.store(g, m, n, acc[i][j]);
        }
}

template <class Op>
inline cudaError_t launch_simt_gemm(const Op &op, int groups, cudaStream_t stream) {
    if (op.M <= 0 || op.N <= 0 || groups <= 0) return cudaSuccess;
    dim3 grid((op.N + kSimtBN - 1) / kSimtBN, (op.M + kSimtBM - 1) / kSimtBM, groups);
    simt_gemm_kernel<Op><<<grid, kSimtThreads, 0, stream>>>(op);
    note_launches(1);
    return cudaGetLastError();
}

}  // namespace mosa
