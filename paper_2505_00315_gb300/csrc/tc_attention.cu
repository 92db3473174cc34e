// Index-masked causal attention over the k selected tokens of each head on
// the tcgen05 tensor cores (Sec. 2.1 Eq. attention with the MoSA mask of
// Sec. 2.2; with I strictly ascending, I_i >= I_j is j <= i).
//
// Forward (F4), one CTA per (128-query tile, sequence b, head h):
//   for each 64-key block j (causal: up to the tile's last query)
//     S_j  = Q K_j^T                       tcgen05, fp32 in TMEM
//     P_j  = exp(S_j/sqrt(h') - m), online max m and sum l per row (4 warps)
//     O_j  = P_j V_j                       tcgen05, P from shared memory
//     o    = o * exp(m_old - m_new) + O_j  (registers)
//   A = o / l, AR = r A, lse = m + log l.
// Q, K, V, P are bf16 hi/lo pairs (v ~ hi + lo), so each product is three
// bf16 MMAs (hi*hi + hi*lo + lo*hi) into one fp32 accumulator, which keeps the
// result at fp32-level accuracy.
// Warp roles: 0 TMA producer, 1 MMA issuer, 2 TMEM allocator, 4-7 softmax
// (one query row per thread).  All waits are bounded.
#include <cudaTypedefs.h>

#include <mutex>

#include "launch.h"
#include "profile.h"
#include "tc_common.cuh"

namespace mosa {
namespace {

using namespace tc;

constexpr int kQ = 128;          // queries per CTA
constexpr int kKV = 64;          // keys per block
constexpr int kThreads = 256;
constexpr int kQBytes = kQ * 64 * 2;    // one half (hi or lo) of the Q tile, 16 KB
constexpr int kKVBytes = kKV * 64 * 2;  // one half of a K or V block, 8 KB
constexpr int kPBytes = kQ * kKV * 2;   // one half of the P tile, 16 KB
constexpr int kStages = 2;

struct FwdSmem {
    // all tiles 1024-byte aligned: 128-byte swizzle atoms
    uint8_t q[2][kQBytes];                   // hi, lo
    uint8_t k[kStages][2][kKVBytes];
    uint8_t v[kStages][2][kKVBytes];
    uint8_t p[2][kPBytes];                   // hi, lo
    uint64_t q_full, kv_full[kStages], kv_empty[kStages], s_full, o_full, p_ready;
    uint32_t tmem;
    int abort;
};

constexpr int kFwdSmem = (int)sizeof(FwdSmem) + 1024;

struct AttnParams {
    CUtensorMap mQ, mK, mV;   // 4-D maps over [H, B, k, 128] pairs, box {64, rows, 1, 1}
    int k, B, Mtok;
    float scale_log2;         // log2(e) / sqrt(h')
    const float *rsel;        // [H, B*k]
    float *A;                 // [H, B*k, 64]
    bf16 *AR;                 // [H, B*k, 128] pair
    float *lse;               // [H, B*k]
    uint32_t *status;
};

__device__ __forceinline__ void flag_timeout(FwdSmem &sm, uint32_t *status) {
    atomicOr(status, kStatusTimeout);
    *(volatile int *)&sm.abort = 1;
}

// Writes 64 values of one row of a K-major, 128-byte-swizzled bf16 tile as
// hi and lo halves (row r of a tile whose rows are 128 bytes).
__device__ __forceinline__ void write_pair_row64(uint8_t *hi_tile, uint8_t *lo_tile, int r,
                                                 const float *v) {
#pragma unroll
    for (int c = 0; c < 8; ++c) {
        uint32_t h4[4], l4[4];
#pragma unroll
        for (int e = 0; e < 4; ++e) {
            const float a = v[c * 8 + 2 * e], b = v[c * 8 + 2 * e + 1];
            const bf16 ha = __float2bfloat16_rn(a), hb = __float2bfloat16_rn(b);
            const bf16 la = __float2bfloat16_rn(a - __bfloat162float(ha));
            const bf16 lb = __float2bfloat16_rn(b - __bfloat162float(hb));
            h4[e] = (uint32_t)__bfloat16_as_ushort(ha) | ((uint32_t)__bfloat16_as_ushort(hb) << 16);
            l4[e] = (uint32_t)__bfloat16_as_ushort(la) | ((uint32_t)__bfloat16_as_ushort(lb) << 16);
        }
        const int off = r * 128 + ((c ^ (r & 7)) << 4);
        *reinterpret_cast<uint4 *>(hi_tile + off) = make_uint4(h4[0], h4[1], h4[2], h4[3]);
        *reinterpret_cast<uint4 *>(lo_tile + off) = make_uint4(l4[0], l4[1], l4[2], l4[3]);
    }
}

__global__ void __launch_bounds__(kThreads, 1) attn_fwd_tc_kernel(const __grid_constant__ AttnParams p) {
    extern __shared__ uint8_t smem_raw[];
    FwdSmem &sm = *reinterpret_cast<FwdSmem *>(
        (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int qt = blockIdx.x, b = blockIdx.y, h = blockIdx.z;
    const int i0 = qt * kQ;
    const int q_end = min(p.k, i0 + kQ);               // exclusive
    const int nblk = (q_end + kKV - 1) / kKV;          // causal: keys < q_end

    if (threadIdx.x == 0) {
        mbar_init(smem_u32(&sm.q_full), 1);
        for (int s = 0; s < kStages; ++s) {
            mbar_init(smem_u32(&sm.kv_full[s]), 1);
            mbar_init(smem_u32(&sm.kv_empty[s]), 1);
        }
        mbar_init(smem_u32(&sm.s_full), 1);
        mbar_init(smem_u32(&sm.o_full), 1);
        mbar_init(smem_u32(&sm.p_ready), 128);
        sm.abort = 0;
        fence_barrier_init();
    }
    if (warp == 2) {
        tmem_alloc(smem_u32(&sm.tmem), 128);
        tmem_relinquish();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = sm.tmem;
    const uint32_t tS = tmem, tO = tmem + 64;

    if (warp == 0) {
        // ---------------------------------------------------------- producer
        if (lane == 0) {
            const uint32_t qb = smem_u32(&sm.q_full);
            mbar_expect_tx(qb, 2 * kQBytes);
            tma_load_4d(smem_u32(sm.q[0]), &p.mQ, qb, 0, i0, b, h);
            tma_load_4d(smem_u32(sm.q[1]), &p.mQ, qb, 64, i0, b, h);
            int issued = 0;
            for (int j = 0; j < nblk; ++j) {
                const int s = j % kStages;
                if (!mbar_wait(smem_u32(&sm.kv_empty[s]), ((j / kStages) & 1) ^ 1) ||
                    *(volatile int *)&sm.abort) {
                    flag_timeout(sm, p.status);
                    break;
                }
                const uint32_t fb = smem_u32(&sm.kv_full[s]);
                mbar_expect_tx(fb, 4 * kKVBytes);
                tma_load_4d(smem_u32(sm.k[s][0]), &p.mK, fb, 0, j * kKV, b, h);
                tma_load_4d(smem_u32(sm.k[s][1]), &p.mK, fb, 64, j * kKV, b, h);
                tma_load_4d(smem_u32(sm.v[s][0]), &p.mV, fb, 0, j * kKV, b, h);
                tma_load_4d(smem_u32(sm.v[s][1]), &p.mV, fb, 64, j * kKV, b, h);
                issued = j + 1;
            }
            if (*(volatile int *)&sm.abort) {
                mbar_wait(qb, 0);
                for (int j = max(0, issued - kStages); j < issued; ++j)
                    mbar_wait(smem_u32(&sm.kv_full[j % kStages]), (j / kStages) & 1);
            }
        }
    } else if (warp == 1) {
        // ------------------------------------------------------------- MMA
        if (lane == 0) {
            constexpr uint32_t idS = idesc_bf16(kQ, kKV, false, false);   // Q (K-major) x K^T (K-major)
            constexpr uint32_t idO = idesc_bf16(kQ, 64, false, true);     // P (K-major) x V (MN-major)
            bool ok = mbar_wait(smem_u32(&sm.q_full), 0);
            const uint32_t q0 = smem_u32(sm.q[0]), q1 = smem_u32(sm.q[1]);
            const uint32_t p0 = smem_u32(sm.p[0]), p1 = smem_u32(sm.p[1]);
            // PV of block j: O = Ph Vh + Ph Vl + Pl Vh
            auto issue_pv = [&](int j) {
                const int s = j % kStages;
                const uint32_t v0 = smem_u32(sm.v[s][0]), v1 = smem_u32(sm.v[s][1]);
                const uint32_t pa[3] = {p0, p0, p1}, vb[3] = {v0, v1, v0};
#pragma unroll
                for (int t = 0; t < 3; ++t)
#pragma unroll
                    for (int kk = 0; kk < kKV / 16; ++kk)
                        mma_bf16(tO, smem_desc_sw128(pa[t] + kk * 32, 16, 1024),
                                 smem_desc_sw128(vb[t] + kk * 2048, kKVBytes, 1024), idO,
                                 (t > 0 || kk > 0) ? 1u : 0u);
                mma_commit(smem_u32(&sm.o_full));
                mma_commit(smem_u32(&sm.kv_empty[s]));
            };
            for (int j = 0; ok && j < nblk; ++j) {
                if (j > 0) {
                    if (!mbar_wait(smem_u32(&sm.p_ready), (j - 1) & 1) || *(volatile int *)&sm.abort) {
                        ok = false;
                        break;
                    }
                    tc_fence_after();
                    issue_pv(j - 1);
                }
                const int s = j % kStages;
                if (!mbar_wait(smem_u32(&sm.kv_full[s]), (j / kStages) & 1)) {
                    ok = false;
                    break;
                }
                tc_fence_after();
                const uint32_t k0 = smem_u32(sm.k[s][0]), k1 = smem_u32(sm.k[s][1]);
                const uint32_t qa[3] = {q0, q0, q1}, kb[3] = {k0, k1, k0};
#pragma unroll
                for (int t = 0; t < 3; ++t)
#pragma unroll
                    for (int kk = 0; kk < 64 / 16; ++kk)
                        mma_bf16(tS, smem_desc_sw128(qa[t] + kk * 32, 16, 1024),
                                 smem_desc_sw128(kb[t] + kk * 32, 16, 1024), idS,
                                 (t > 0 || kk > 0) ? 1u : 0u);
                mma_commit(smem_u32(&sm.s_full));
            }
            if (ok && nblk > 0) {
                if (mbar_wait(smem_u32(&sm.p_ready), (nblk - 1) & 1) && !*(volatile int *)&sm.abort) {
                    tc_fence_after();
                    issue_pv(nblk - 1);
                } else {
                    ok = false;
                }
            }
            if (!ok) {
                flag_timeout(sm, p.status);
                // release the softmax warps
                mma_commit(smem_u32(&sm.s_full));
                mma_commit(smem_u32(&sm.o_full));
            }
        }
    } else if (warp >= 4) {
        // ---------------------------------------------------------- softmax
        const int q = warp - 4;
        const int r = q * 32 + lane;
        const int i = i0 + r;
        const uint32_t lane_off = (uint32_t)(q * 32) << 16;
        float o[64];
#pragma unroll
        for (int c = 0; c < 64; ++c) o[c] = 0.f;
        float m = -INFINITY, l = 0.f, corr_prev = 1.f;
        bool ok = true;
        for (int j = 0; j < nblk; ++j) {
            if (!mbar_wait(smem_u32(&sm.s_full), j & 1) || *(volatile int *)&sm.abort) {
                ok = false;
                break;
            }
            tc_fence_after();
            float s[64];
            {
                float t32[32];
                tmem_ld32(tS + lane_off, t32);
#pragma unroll
                for (int c = 0; c < 32; ++c) s[c] = t32[c];
                tmem_ld32(tS + lane_off + 32, t32);
#pragma unroll
                for (int c = 0; c < 32; ++c) s[32 + c] = t32[c];
            }
            const int j0 = j * kKV;
            float mx = m;
#pragma unroll
            for (int c = 0; c < 64; ++c) {
                s[c] = (j0 + c <= i) ? s[c] * p.scale_log2 : -INFINITY;
                mx = fmaxf(mx, s[c]);
            }
            const float corr = exp2f(m - mx);   // 0 on the first block (m = -inf)
            float sum = 0.f;
#pragma unroll
            for (int c = 0; c < 64; ++c) {
                s[c] = exp2f(s[c] - mx);
                sum += s[c];
            }
            l = l * corr + sum;
            m = mx;
            if (j > 0) {
                // O of the previous block: it is relative to the previous max.
                if (!mbar_wait(smem_u32(&sm.o_full), (j - 1) & 1)) {
                    ok = false;
                    break;
                }
                tc_fence_after();
                float t32[32];
                tmem_ld32(tO + lane_off, t32);
#pragma unroll
                for (int c = 0; c < 32; ++c) o[c] = o[c] * corr_prev + t32[c];
                tmem_ld32(tO + lane_off + 32, t32);
#pragma unroll
                for (int c = 0; c < 32; ++c) o[32 + c] = o[32 + c] * corr_prev + t32[c];
            }
            corr_prev = corr;
            write_pair_row64(sm.p[0], sm.p[1], r, s);
            fence_proxy_async();
            tc_fence_before();
            mbar_arrive(smem_u32(&sm.p_ready));
        }
        if (ok && nblk > 0) {
            if (mbar_wait(smem_u32(&sm.o_full), (nblk - 1) & 1)) {
                tc_fence_after();
                float t32[32];
                tmem_ld32(tO + lane_off, t32);
#pragma unroll
                for (int c = 0; c < 32; ++c) o[c] = o[c] * corr_prev + t32[c];
                tmem_ld32(tO + lane_off + 32, t32);
#pragma unroll
                for (int c = 0; c < 32; ++c) o[32 + c] = o[32 + c] * corr_prev + t32[c];
            } else {
                ok = false;
            }
        }
        if (!ok) flag_timeout(sm, p.status);
        if (ok && i < p.k && !*(volatile int *)&sm.abort) {
            const size_t row = (size_t)h * p.Mtok + (size_t)b * p.k + i;
            const float inv = 1.f / l;
            const float rr = p.rsel[row];
            float *arow = p.A + row * 64;
#pragma unroll
            for (int c = 0; c < 64; c += 4)
                *reinterpret_cast<float4 *>(arow + c) =
                    make_float4(o[c] * inv, o[c + 1] * inv, o[c + 2] * inv, o[c + 3] * inv);
            bf16 *ar = p.AR + row * 128;
#pragma unroll
            for (int c = 0; c < 64; c += 8) {
                uint32_t h4[4], l4[4];
#pragma unroll
                for (int e = 0; e < 4; ++e) {
                    const float a = rr * o[c + 2 * e] * inv, bb = rr * o[c + 2 * e + 1] * inv;
                    const bf16 ha = __float2bfloat16_rn(a), hb = __float2bfloat16_rn(bb);
                    const bf16 la = __float2bfloat16_rn(a - __bfloat162float(ha));
                    const bf16 lb = __float2bfloat16_rn(bb - __bfloat162float(hb));
                    h4[e] = (uint32_t)__bfloat16_as_ushort(ha) | ((uint32_t)__bfloat16_as_ushort(hb) << 16);
                    l4[e] = (uint32_t)__bfloat16_as_ushort(la) | ((uint32_t)__bfloat16_as_ushort(lb) << 16);
                }
                *reinterpret_cast<uint4 *>(ar + c) = make_uint4(h4[0], h4[1], h4[2], h4[3]);
                *reinterpret_cast<uint4 *>(ar + 64 + c) = make_uint4(l4[0], l4[1], l4[2], l4[3]);
            }
            // lse in natural-log units of the scaled scores
            p.lse[row] = (m + log2f(l)) * 0.69314718055994531f;
        }
    }
    tc_fence_before();
    __syncthreads();
    if (warp == 2) {
        tc_fence_after();
        tmem_dealloc(tmem, 128);
    }
}

PFN_cuTensorMapEncodeTiled_v12000 encode() {
    static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
    static std::once_flag once;
    std::call_once(once, [] {
        void *ptr = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &ptr, 12000,
                                             cudaEnableDefault, &q) == cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(ptr);
    });
    return fn;
}

// [H, B, k, 128] bf16 pair array (row = 64 hi + 64 lo), box {64, rows, 1, 1}:
// rows past k of one sequence read as zeros.
bool map_units(CUtensorMap *m, const void *base, int H, int B, int k, uint32_t rows) {
    auto fn = encode();
    if (!fn) return false;
    const cuuint64_t dims[4] = {128, (cuuint64_t)k, (cuuint64_t)B, (cuuint64_t)H};
    const cuuint64_t strides[3] = {256, (cuuint64_t)k * 256, (cuuint64_t)B * k * 256};
    const cuuint32_t box[4] = {64, rows, 1, 1}, es[4] = {1, 1, 1, 1};
    return fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 4, const_cast<void *>(base), dims, strides, box,
              es, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
              CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

}  // namespace

cudaError_t tc_attn_fwd(const Dims &dm, const Saved &sv, cudaStream_t s) {
    AttnParams p;
    memset(&p, 0, sizeof(p));
    bool ok = map_units(&p.mQ, sv.Q, dm.H, dm.B, dm.k, kQ) &&
              map_units(&p.mK, sv.K, dm.H, dm.B, dm.k, kKV) &&
              map_units(&p.mV, sv.V, dm.H, dm.B, dm.k, kKV);
    if (!ok) return cudaErrorInvalidValue;
    p.k = dm.k;
    p.B = dm.B;
    p.Mtok = dm.B * dm.k;
    p.scale_log2 = 1.4426950408889634f / sqrtf(64.f);
    p.rsel = sv.rsel;
    p.A = sv.A;
    p.AR = static_cast<bf16 *>(sv.AR);
    p.lse = sv.lse;
    p.status = sv.status;
    static std::once_flag once;
    static cudaError_t attr = cudaSuccess;
    std::call_once(once, [] {
        attr = cudaFuncSetAttribute(attn_fwd_tc_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                    kFwdSmem);
    });
    if (attr != cudaSuccess) return attr;
    dim3 grid((dm.k + kQ - 1) / kQ, dm.B, dm.H);
    attn_fwd_tc_kernel<<<grid, kThreads, kFwdSmem, s>>>(p);
    note_launches(1);
    return cudaGetLastError();
}

}  // namespace mosa
