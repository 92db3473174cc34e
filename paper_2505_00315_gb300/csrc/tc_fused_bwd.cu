// Fused backward of the selected-token path for k <= 128 (Sec. 2.2, Eq.
// mosa_mha, differentiated with I held fixed): one CTA per 128-row tile of one
// head (U = floor(128 / k) sequences, as in the fused forward), all products
// on the tensor cores with fp32 accumulators in TMEM:
//   phase 1  G = dY[g(m), :] W_o[h]^T        K = d in 64-wide blocks, a 3-stage
//            ring: W_o blocks by TMA, the selected rows of dY by cp.async
//   phase 2  D = <AR, G> = r <A, G>, dA = r G (bf16 pair, shared memory),
//            dlogit = D (1 - r) (the router gradient through diag(r))
//   phase 3  S = Q K^T, dP = dA V^T; P from the saved log-sum-exp; dV = P^T dA;
//            dS = P o (dP - D); dK = dS^T Q / sqrt(h'), dQ = dS K / sqrt(h')
//   phase 4  dQ|dK|dV (and dlogit) to global memory for dX and the weight
//            gradients.
// dX (tc_dx.cu) and the weight gradients, which reduce over all tiles of a
// head, stay separate products (dW_o, dW_q|dW_k|dW_v|dW_r in tc_gemm.cu).
//
// Warps: 0 TMA producer, 1 MMA issuer, 2 TMEM owner, 3 idle; 4-11 gather,
// row terms, softmax passes and epilogues, two per TMEM lane quadrant.
// Every wait is bounded.
#include <mutex>

#include "launch.h"
#include "profile.h"
#include "tc_common.cuh"
#include "tc_tiles.cuh"
#include "tmap.h"

namespace mosa {
namespace {

using namespace tc;

constexpr int kThreads = 384;
constexpr int kWorkers = 256;
constexpr int kStages = 3;
constexpr int kHalf = kTileHalf;                 // 16 KB
constexpr int kStageBytes = kHalf + 8192;        // gathered dY block + W_o block

// TMEM columns
constexpr uint32_t kColG = 0, kColS = 64, kColDP = 192, kColDV = 320, kColDK = 384, kColDQ = 448;

struct FusedBwdSmem {
    // phase 1: the ring (3 x 24 KB); phase 3: P / dS pair tile [half][key block]
    // (64 KB)
    uint8_t r1[5 * kHalf];
    uint8_t da[2][kHalf];        // dA pair; phase 4: epilogue staging (8 x 4 KB)
    uint8_t qkv[3][2][kHalf];    // Q, K, V pairs
    float part[2][128];          // partial <A, G> per column half
    float Dd[128];               // D per tile row
    int rows[128];               // b*T + I of each tile row, -1 outside the tile's sequences
    uint64_t full[kStages], empty[kStages];
    uint64_t qkv_full, g_done, da_ready, sp_full, p_ready, pv_done, ds_ready, acc_done;
    uint32_t tmem;
    int abort;
};
constexpr int kSmem = (int)sizeof(FusedBwdSmem) + 1024;
static_assert(kSmem <= 227 * 1024, "shared memory");
static_assert(kStages * kStageBytes <= 5 * kHalf, "region 1");

struct FusedBwdParams {
    CUtensorMap mWo;       // W_o: [H, 64, d], box {64, 64, 1}
    CUtensorMap mQKV[3];   // Q, K, V pairs: [H, B*k, 128], box {64, 128, 1}
    const bf16 *dY;        // [B*T, d]
    const int32_t *gidx;   // [H, B*k]
    const float *rsel;     // [H, B*k]
    const bf16 *AR;        // [H, B*k, 128] pair of AR = diag(r) A
    const float *lse;      // [H, B*k]
    bf16 *dQKV;            // [H, B*k, 512] pair: dQ|dK|dV|dlogit hi, then lo
    float *Dd, *dlogit;    // [H, B*k]
    int B, T, d, k, U, Mtok;
    float scale, scale_log2;
    uint32_t *status;
    unsigned long long *span;   // measurement: kernel span slot, or null
};

__device__ __forceinline__ bool wait_or_abort(FusedBwdSmem &sm, uint64_t &bar, uint32_t parity,
                                              uint32_t *status) {
    if (*(volatile int *)&sm.abort) return false;
    if (mbar_wait(smem_u32(&bar), parity)) return true;
    atomicOr(status, kStatusTimeout);
    *(volatile int *)&sm.abort = 1;
    return false;
}

__global__ void __launch_bounds__(kThreads, 1) fused_bwd_kernel(const __grid_constant__ FusedBwdParams p) {
    extern __shared__ uint8_t smem_raw[];
    FusedBwdSmem &sm = *reinterpret_cast<FusedBwdSmem *>(
        (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int b0 = blockIdx.x * p.U, h = blockIdx.y;
    const int nkb = (p.d + 63) / 64;
    const size_t row_base = (size_t)h * p.Mtok + (size_t)b0 * p.k;
    uint8_t(*ptile)[2][kHalf] = reinterpret_cast<uint8_t(*)[2][kHalf]>(&sm.r1[0]);
    auto ring = [&](int s) -> uint8_t * { return &sm.r1[0] + s * kStageBytes; };

    if (threadIdx.x == 0) {
        for (int s = 0; s < kStages; ++s) {
            mbar_init(smem_u32(&sm.full[s]), 1 + kWorkers);
            mbar_init(smem_u32(&sm.empty[s]), 1);
        }
        mbar_init(smem_u32(&sm.qkv_full), 1);
        mbar_init(smem_u32(&sm.g_done), 1);
        mbar_init(smem_u32(&sm.da_ready), kWorkers);
        mbar_init(smem_u32(&sm.sp_full), 1);
        mbar_init(smem_u32(&sm.p_ready), kWorkers);
        mbar_init(smem_u32(&sm.pv_done), 1);
        mbar_init(smem_u32(&sm.ds_ready), kWorkers);
        mbar_init(smem_u32(&sm.acc_done), 1);
        sm.abort = 0;
        fence_barrier_init();
    }
    if (warp == 2) {
        tmem_alloc(smem_u32(&sm.tmem), 512);
        tmem_relinquish();
    }
    pdl_wait();  // everything read below was written by earlier kernels
    span_begin(p.span);
    if (threadIdx.x < 128) {
        const int r = threadIdx.x, u = r / p.k;
        const bool valid = u < p.U && b0 + u < p.B;
        sm.rows[r] = valid ? p.gidx[row_base + r] : -1;
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = sm.tmem;

    if (warp == 0) {
        // ---------------------------------------------------------- producer
        if (lane == 0) {
            // Q, K, V pairs of the tile (rows past B*k read as zeros)
            const uint32_t qb = smem_u32(&sm.qkv_full);
            mbar_expect_tx(qb, 6 * kHalf);
            for (int j = 0; j < 3; ++j)
                for (int hf = 0; hf < 2; ++hf)
                    tma_load_3d(smem_u32(sm.qkv[j][hf]), &p.mQKV[j], qb, 64 * hf, b0 * p.k, h);
            // phase 1: W_o blocks (rows p, 64 columns of d)
            int issued = 0;
            for (int kb = 0; kb < nkb; ++kb) {
                const int s = kb % kStages;
                if (!wait_or_abort(sm, sm.empty[s], ((kb / kStages) & 1) ^ 1, p.status)) break;
                const uint32_t fb = smem_u32(&sm.full[s]);
                mbar_expect_tx(fb, 8192);
                tma_load_3d(smem_u32(ring(s) + kHalf), &p.mWo, fb, kb * 64, 0, h);
                issued = kb + 1;
            }
            // drain: Q, K, V and the last load of every ring slot have landed (a
            // stage whose gathering threads gave up before issuing it never
            // completes; its wait then runs out the full bound)
            drain_phase(qb, 0);
            for (int kb = max(0, issued - kStages); kb < issued; ++kb)
                drain_phase(smem_u32(&sm.full[kb % kStages]), (kb / kStages) & 1);
        }
    } else if (warp == 1) {
        // ------------------------------------------------------------- MMA
        if (lane == 0) {
            bool ok = true;
            // phase 1: G = dY[I] W_o^T into TMEM 0..63 (both operands K-major)
            constexpr uint32_t idG = idesc_bf16(128, 64, false, false);
            for (int kb = 0; kb < nkb && ok; ++kb) {
                const int s = kb % kStages;
                if (!(ok = wait_or_abort(sm, sm.full[s], (kb / kStages) & 1, p.status))) break;
                tc_fence_after();
                const uint32_t a = smem_u32(ring(s)), b = a + kHalf;
#pragma unroll
                for (int j = 0; j < 4; ++j)
                    mma_bf16(tmem + kColG, smem_desc_sw128(a + j * 32, 16, 1024),
                             smem_desc_sw128(b + j * 32, 16, 1024), idG, (kb > 0 || j > 0) ? 1u : 0u);
                mma_commit(smem_u32(&sm.empty[s]));
            }
            mma_commit(smem_u32(&sm.g_done));
            // phase 3
            constexpr uint32_t idKK = idesc_bf16(128, 128, false, false);  // S, dP
            constexpr uint32_t idMN = idesc_bf16(128, 64, true, true);     // dV, dK
            constexpr uint32_t idKM = idesc_bf16(128, 64, false, true);    // dQ
            const uint32_t q0 = smem_u32(sm.qkv[0][0]), q1 = smem_u32(sm.qkv[0][1]);
            const uint32_t k0 = smem_u32(sm.qkv[1][0]), k1 = smem_u32(sm.qkv[1][1]);
            const uint32_t v0 = smem_u32(sm.qkv[2][0]), v1 = smem_u32(sm.qkv[2][1]);
            const uint32_t a0 = smem_u32(sm.da[0]), a1 = smem_u32(sm.da[1]);
            ok = ok && wait_or_abort(sm, sm.qkv_full, 0, p.status);
            if (ok) {
                tc_fence_after();
                mma_pair3(tmem + kColS, q0, q1, k0, k1, false, false, idKK, false);   // S = Q K^T
            }
            ok = ok && wait_or_abort(sm, sm.da_ready, 0, p.status);
            if (ok) {
                tc_fence_after();
                mma_pair3(tmem + kColDP, a0, a1, v0, v1, false, false, idKK, false);  // dP = dA V^T
            }
            mma_commit(smem_u32(&sm.sp_full));
            ok = ok && wait_or_abort(sm, sm.p_ready, 0, p.status);
            if (ok) {
                tc_fence_after();
                mma_k128(tmem + kColDV, ptile, sm.da, true, idMN);   // dV = P^T dA
            }
            mma_commit(smem_u32(&sm.pv_done));
            ok = ok && wait_or_abort(sm, sm.ds_ready, 0, p.status);
            if (ok) {
                tc_fence_after();
                mma_k128(tmem + kColDK, ptile, sm.qkv[0], true, idMN);    // dK = dS^T Q
                mma_k128(tmem + kColDQ, ptile, sm.qkv[1], false, idKM);   // dQ = dS K
            }
            if (!ok) {
                // release every wait of the other warps that may still be pending
                mma_commit(smem_u32(&sm.sp_full));
                mma_commit(smem_u32(&sm.pv_done));
            }
            drain_mmas(smem_u32(&sm.acc_done));   // acc_done's only phase covers every MMA
        }
    } else if (warp >= 4) {
        const int t = threadIdx.x - 128;
        const int q = warp & 3, ch = (warp - 4) >> 2;
        const int r = q * 32 + lane;
        const uint32_t lane_off = (uint32_t)(q * 32) << 16;
        const TileRow tr = tile_row(r, p.k, p.U, b0, p.B);
        const bool valid = tr.valid;
        const int lo = tr.lo;
        const unsigned vmask = __ballot_sync(0xffffffffu, valid);
        const size_t grow = row_base + r;   // head row of this thread's tile row
        const size_t grow0 = row_base + q * 32;

        // ------------------------------------------- phase 1: gather dY rows
        {
            const int chunk = t & 7, sub = t >> 3;
            int landed = 0, issued = 0;
            for (int kb = 0; kb < nkb; ++kb) {
                const int s = kb % kStages;
                if (!wait_or_abort(sm, sm.empty[s], ((kb / kStages) & 1) ^ 1, p.status)) break;
                const uint32_t a = smem_u32(ring(s));
                const int col = kb * 64 + chunk * 8;
#pragma unroll
                for (int j = 0; j < 4; ++j) {
                    const int row = sub + 32 * j;
                    const int src = sm.rows[row];
                    const uint32_t nbytes = (src >= 0 && col < p.d) ? 16u : 0u;
                    const bf16 *g = p.dY + (size_t)(src >= 0 ? src : 0) * p.d + (nbytes ? col : 0);
                    cp_async16(a + row * 128 + ((chunk ^ (row & 7)) << 4), g, nbytes);
                }
                cp_async_commit();
                issued = kb + 1;
                if (kb >= 1) {
                    cp_async_wait<1>();
                    fence_proxy_async();
                    mbar_arrive(smem_u32(&sm.full[(kb - 1) % kStages]));
                    ++landed;
                }
            }
            cp_async_wait<0>();
            fence_proxy_async();
            for (int kb = landed; kb < issued; ++kb) mbar_arrive(smem_u32(&sm.full[kb % kStages]));
        }

        // ----------------------------------------------- phase 2: row terms
        bool ok = wait_or_abort(sm, sm.g_done, 0, p.status);
        tc_fence_after();
        float g[32];
        tmem_ld32(tmem + kColG + lane_off + 32 * ch, g);   // G columns 32 ch .. +31
        float dd = 0.f;   // this half of D = <AR, G> = r <A, G>
        if (valid) {
            // columns 32 ch .. +31 of the AR pair row: hi at 32 ch, lo at 64 + 32 ch
            const uint4 *hrow = reinterpret_cast<const uint4 *>(p.AR + grow * 128 + 32 * ch);
            const uint4 *lrow = reinterpret_cast<const uint4 *>(p.AR + grow * 128 + 64 + 32 * ch);
#pragma unroll
            for (int u = 0; u < 4; ++u) dd = dot_pair8(hrow[u], lrow[u], g + 8 * u, dd);
        }
        const float rr = valid ? p.rsel[grow] : 0.f;
        put_pair32(sm.da[0], sm.da[1], r, 32 * ch, g, rr);   // dA = r G
        sm.part[ch][r] = dd;
        fence_proxy_async();
        tc_fence_before();
        named_barrier(1, kWorkers);
        dd = sm.part[0][r] + sm.part[1][r];          // D = rowsum(dA o A)
        const float dlg = dd * (1.f - rr);           // dlogit = r (1 - r) <A, G>
        if (ch == 0) {
            sm.Dd[r] = dd;
            if (ok && valid) {
                p.Dd[grow] = dd;
                p.dlogit[grow] = dlg;
                // dlogit as column 192 (hi) / 448 (lo) of the dQKV pair row: column
                // 0 of the block the dW product reads for dW_r (its other columns
                // only reach accumulator columns that are never read)
                const bf16 dh = __float2bfloat16_rn(dlg);
                const bf16 dlo = __float2bfloat16_rn(dlg - __bfloat162float(dh));
                p.dQKV[grow * 512 + 192] = dh;
                p.dQKV[grow * 512 + 448] = dlo;
            }
        }
        mbar_arrive(smem_u32(&sm.da_ready));

        // ------------------------------------------- phase 3: P and dS passes
        const int cb = 64 * ch;
        const float l2 = valid ? p.lse[grow] * 1.4426950408889634f : 0.f;
        ok = wait_or_abort(sm, sm.sp_full, 0, p.status) && ok;
        tc_fence_after();
#pragma unroll 1
        for (int c0 = cb; c0 < cb + 64; c0 += 32) {
            float t32[32];
            tmem_ld32(tmem + kColS + lane_off + c0, t32);
#pragma unroll
            for (int c = 0; c < 32; ++c)
                t32[c] = (valid && c0 + c <= r && c0 + c >= lo) ? exp2_fast(t32[c] * p.scale_log2 - l2) : 0.f;
            write_pair32(ptile, r, c0, t32);
        }
        fence_proxy_async();
        tc_fence_before();
        mbar_arrive(smem_u32(&sm.p_ready));
        ok = wait_or_abort(sm, sm.pv_done, 0, p.status) && ok;   // P read by dV: overwrite with dS
        tc_fence_after();
#pragma unroll 1
        for (int c0 = cb; c0 < cb + 64; c0 += 32) {
            float t32[32], d32[32];
            tmem_ld32(tmem + kColS + lane_off + c0, t32);
            tmem_ld32(tmem + kColDP + lane_off + c0, d32);
#pragma unroll
            for (int c = 0; c < 32; ++c) {
                const float pr = (valid && c0 + c <= r && c0 + c >= lo) ? exp2_fast(t32[c] * p.scale_log2 - l2) : 0.f;
                t32[c] = pr * (d32[c] - dd);
            }
            write_pair32(ptile, r, c0, t32);
        }
        fence_proxy_async();
        tc_fence_before();
        mbar_arrive(smem_u32(&sm.ds_ready));

        // ---------------------------------------------- phase 4: dQ|dK|dV out
        ok = wait_or_abort(sm, sm.acc_done, 0, p.status) && ok;
        tc_fence_after();
        const bool live = __all_sync(0xffffffffu, ok && !*(volatile int *)&sm.abort);
        uint8_t *xb = &sm.da[0][0] + (warp - 4) * 4096;   // dA is no longer read
        {
            const uint32_t src[3] = {kColDQ, kColDK, kColDV};
            const float fac[3] = {p.scale, p.scale, 1.f};
#pragma unroll
            for (int j = 0; j < 3; ++j) {
                float v[32];
                tmem_ld32(tmem + src[j] + lane_off + 32 * ch, v);
                if (live) {
                    stage_pair32(xb, v, fac[j], lane);
                    store_rows128(xb, lane, [&](int rl, int c) -> uint4 * {
                        if (!((vmask >> rl) & 1u)) return nullptr;
                        bf16 *row = p.dQKV + (grow0 + rl) * 512 + 64 * j + 32 * ch;
                        return c < 4 ? reinterpret_cast<uint4 *>(row) + c
                                     : reinterpret_cast<uint4 *>(row + 256) + (c - 4);
                    });
                }
            }
        }
        pdl_trigger();
    }
    tc_fence_before();
    __syncthreads();
    span_end(p.span);
    if (warp == 2) {
        tc_fence_after();
        tmem_dealloc(tmem, 512);
    }
}

bool map3(CUtensorMap *m, const void *base, uint64_t H, uint64_t rows, uint64_t cols,
          uint32_t box_rows) {
    const uint64_t dims[3] = {cols, rows, H}, strides[2] = {cols * 2, rows * cols * 2};
    const uint32_t box[3] = {64, box_rows, 1};
    return tmap_bf16(m, base, 3, dims, strides, box);
}

}  // namespace

// Opt-in (MOSA_FUSED_BWD=1): measured on GB300 the fused kernel beats G plus
// the attention backward as separate kernels, but it holds a whole SM per CTA
// and so cannot overlap dW_o; the separate kernels' schedule (dW_o beside G,
// dX beside dW) finishes the backward sooner at every benchmarked size.
bool use_fused_backward(const Dims &dm) {
    const char *f = std::getenv("MOSA_FUSED_BWD");
    if (f == nullptr || f[0] != '1') return false;
    return use_tc(dm) && dm.k <= 128;
}

cudaError_t tc_fused_backward(const Dims &dm, const void *W_o, const void *dY, const Saved &sv,
                              cudaStream_t s) {
    FusedBwdParams p;
    memset(&p, 0, sizeof(p));
    const int Mtok = dm.B * dm.k;
    const void *QKV[3] = {sv.Q, sv.K, sv.V};
    bool ok = map3(&p.mWo, W_o, dm.H, 64, dm.d, 64);
    for (int j = 0; j < 3; ++j)
        ok = ok && map3(&p.mQKV[j], QKV[j], dm.H, Mtok, 128, 128);
    if (!ok) return cudaErrorInvalidValue;
    p.dY = static_cast<const bf16 *>(dY);
    p.gidx = sv.gidx;
    p.rsel = sv.rsel;
    p.AR = static_cast<const bf16 *>(sv.AR);
    p.lse = sv.lse;
    p.dQKV = static_cast<bf16 *>(sv.dQKV);
    p.Dd = sv.Dd;
    p.dlogit = sv.dlogit;
    p.B = dm.B;
    p.T = dm.T;
    p.d = dm.d;
    p.k = dm.k;
    p.U = 128 / dm.k;
    p.Mtok = Mtok;
    p.scale = 1.f / sqrtf(64.f);
    p.scale_log2 = 1.4426950408889634f / sqrtf(64.f);
    p.status = sv.status;
    p.span = active_span();
    const cudaError_t attr = allow_smem((const void *)fused_bwd_kernel, kSmem);
    if (attr != cudaSuccess) return attr;
    const dim3 grid((dm.B + p.U - 1) / p.U, dm.H);
    cudaError_t e = launch_pdl(fused_bwd_kernel, grid, dim3(kThreads), kSmem, s, p);
    note_launches(1);
    return e;
}

}  // namespace mosa
