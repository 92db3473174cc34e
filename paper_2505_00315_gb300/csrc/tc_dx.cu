// Products whose rows scatter-add into a [B*T, d] array through the selected
// token rows g(m) = b*T + I[b,h,i] of head h (Sec. 2.2, Eq. mosa_mha):
//   input gradient B3 (differentiated through the gather X^s = X[I] and the
//   router r = sigmoid(X W^r)):
//     dX[g(m), n] += sum_j [dQ|dK|dV]_j(m, :) W_j[h](n, :)  +  dlogit(m) W_r[n, h]
//   output F5 (used when the attention runs as its own kernel, k > 128):
//     Y[g(m), n]  += AR(m, :) W_o[h](:, n),   AR = diag(r^topk) A
//
// The work is a list of units (head, 128-row tile, 256-column chunk of d),
// head-major, and a persistent grid of at most one CTA per SM takes a
// contiguous range of it, so every SM gets the same number of units whatever
// the tile count.  A CTA loads a tile's A pairs (dQ|dK|dV, 96 KB, or AR,
// 32 KB) by TMA once for all the chunks it holds of that tile; the weight
// blocks of a chunk (W_j: 256 rows of d x 64; W_o: 64 x 256 columns of d)
// stream through a 3-slot ring; the chunk accumulators alternate between two
// 256-column halves of TMEM, so the scatter-add of one chunk (red.add.v4
// through a per-warp staging buffer; for dX with dlogit x W_r added from an
// fp32 transpose of W_r) runs while the MMAs of the next one do.  Each
// product with a pair operand is two MMAs (hi, lo); on the fp16 attention
// path (k > 128) dX reads dQ|dK|dV as single fp16 values and fp16 copies of
// W_q|W_k|W_v, and Y reads AR as fp16 with an fp16 copy of W_o: one MMA.
// Warps: 0 TMA producer, 1 MMA issuer, 2 TMEM owner, 3 idle, 4-11 epilogue
// (warp w: tile rows 32 (w % 4) .. +31, chunk columns 128 ((w - 4) / 4) ..).
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
constexpr int kChunk = 256;
constexpr int kSlots = 3;
constexpr int kWBytes = 256 * 128;   // one weight block of a chunk: 32 KB

struct DxSmem {
    uint8_t a[3][2][kTileHalf];      // A pairs of the tile [j][hi / lo]: dQ, dK, dV, or AR
    uint8_t w[kSlots][kWBytes];      // weight blocks
    uint8_t stage[8][4096];          // epilogue staging, one buffer per epilogue warp
    uint64_t a_full[3], a_empty[3], w_full[kSlots], w_empty[kSlots], out_full[2], out_empty[2];
    uint64_t drained;   // the MMA issuer's final drain
    uint32_t tmem;
    int abort;
};
constexpr int kSmem = (int)sizeof(DxSmem) + 1024;
static_assert(kSmem <= 227 * 1024, "shared memory");

struct DxParams {
    CUtensorMap mA;       // dX: dQKV pair [H, B*k, 512]; Y: AR pair [H, B*k, 128]; box {64, 128, 1}
    CUtensorMap mW[3];    // dX: W_q, W_k, W_v [H, d, 64], box {64, 256, 1}; Y: W_o [H, 64, d], box {64, 64, 1}
    const int32_t *gidx;  // [H, B*k]
    const float *dlogit;  // [H, B*k] (dX)
    const float *WrT;     // [H, d] fp32 transpose of W_r (dX)
    float *dX;            // [B*T, d] (dX or Y), accumulated into
    int Mtok, d;
    int mt, nch;          // tiles per head, chunks per tile
    long long units;      // H * mt * nch
    uint32_t *status;
    int f16;              // dX: A = fp16 dQKV rows [H, B*k, 256], W = fp16 copies (one MMA);
                          // Y: A = fp16 AR rows [H, B*k, 64], W = the fp16 copy of W_o
    unsigned long long *span;   // measurement: kernel span slot, or null
};

__device__ __forceinline__ bool dwait(DxSmem &sm, uint64_t &bar, uint32_t parity, uint32_t *status) {
    if (*(volatile int *)&sm.abort) return false;
    if (mbar_wait(smem_u32(&bar), parity)) return true;
    atomicOr(status, kStatusTimeout);
    *(volatile int *)&sm.abort = 1;
    return false;
}

// kOut = false: dX (three A matrices, K-major W_j blocks, plus dlogit W_r);
// kOut = true: Y (one A matrix, AR; MN-major W_o chunks).
template <bool kOut>
__global__ void __launch_bounds__(kThreads, 1) scatter_product_kernel(const __grid_constant__ DxParams p) {
    constexpr int NM = kOut ? 1 : 3;          // A matrices per tile
    constexpr int kLo = kOut ? 64 : 256;      // column of the lo half of a pair row
    extern __shared__ uint8_t smem_raw[];
    DxSmem &sm = *reinterpret_cast<DxSmem *>(
        (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    // this CTA's units [u0, u1); unit u = (h * mt + tile) * nch + chunk
    const long long u0 = p.units * blockIdx.x / gridDim.x;
    const long long u1 = p.units * (blockIdx.x + 1) / gridDim.x;
    const int nu = (int)(u1 - u0);

    if (threadIdx.x == 0) {
        for (int j = 0; j < NM; ++j) {
            mbar_init(smem_u32(&sm.a_full[j]), 1);
            mbar_init(smem_u32(&sm.a_empty[j]), 1);
        }
        for (int s = 0; s < kSlots; ++s) {
            mbar_init(smem_u32(&sm.w_full[s]), 1);
            mbar_init(smem_u32(&sm.w_empty[s]), 1);
        }
        for (int i = 0; i < 2; ++i) {
            mbar_init(smem_u32(&sm.out_full[i]), 1);
            mbar_init(smem_u32(&sm.out_empty[i]), kWorkers);
        }
        mbar_init(smem_u32(&sm.drained), 1);
        sm.abort = 0;
        fence_barrier_init();
    }
    if (warp == 2) {
        tmem_alloc(smem_u32(&sm.tmem), 512);
        tmem_relinquish();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = sm.tmem;
    pdl_wait();  // the A pairs (and dlogit) come from earlier kernels
    span_begin(p.span);

    if (warp == 0) {
        if (lane == 0) {
            int ntile = 0;  // tiles started so far
            int nw = 0;     // weight-block loads issued
            int na[3] = {0, 0, 0};   // A_j loads issued
            for (int i = 0; i < nu; ++i) {
                const long long u = u0 + i;
                const int c = (int)(u % p.nch);
                const long long tile = u / p.nch;
                const int h = (int)(tile / p.mt), m0 = (int)(tile % p.mt) * 128;
                const bool fresh = i == 0 || c == 0;
                bool ok = true;
                for (int j = 0; j < NM; ++j) {
                    const int idx = NM * i + j, s = idx % kSlots;
                    if (!(ok = dwait(sm, sm.w_empty[s], ((idx / kSlots) & 1) ^ 1, p.status))) break;
                    if (fresh) {
                        // A_j of the previous tile frees once its last j-products end
                        if (ntile > 0 && !(ok = dwait(sm, sm.a_empty[j], (ntile - 1) & 1, p.status)))
                            break;
                        const uint32_t ab = smem_u32(&sm.a_full[j]);
                        mbar_expect_tx(ab, (p.f16 ? 1 : 2) * kTileHalf);
                        tma_load_3d(smem_u32(sm.a[j][0]), &p.mA, ab, 64 * j, m0, h);        // hi
                        if (!p.f16)
                            tma_load_3d(smem_u32(sm.a[j][1]), &p.mA, ab, kLo + 64 * j, m0, h);  // lo
                        ++na[j];
                    }
                    const uint32_t fb = smem_u32(&sm.w_full[s]);
                    mbar_expect_tx(fb, kWBytes);
                    if (kOut) {
                        // W_o rows 0..63 (K), columns c*256 .. +255 (N) as four 64-wide blocks
                        for (int q = 0; q < 4; ++q)
                            tma_load_3d(smem_u32(sm.w[s]) + q * 8192, &p.mW[0], fb, c * kChunk + 64 * q, 0, h);
                    } else {
                        tma_load_3d(smem_u32(sm.w[s]), &p.mW[j], fb, 0, c * kChunk, h);
                    }
                    nw = idx + 1;
                }
                if (!ok) break;
                if (fresh) ++ntile;
            }
            // drain: the last load of every weight slot and of every A_j has landed
            for (int idx = max(0, nw - kSlots); idx < nw; ++idx)
                drain_phase(smem_u32(&sm.w_full[idx % kSlots]), (idx / kSlots) & 1);
            for (int j = 0; j < NM; ++j)
                if (na[j] > 0) drain_phase(smem_u32(&sm.a_full[j]), (na[j] - 1) & 1);
        }
    } else if (warp == 1) {
        if (lane == 0) {
            // B: W_j blocks K-major (dX), W_o chunks MN-major (Y)
            const uint32_t idX = p.f16 ? idesc_f16(128, kChunk, false, kOut)
                                       : idesc_bf16(128, kChunk, false, kOut);
            const int halves = p.f16 ? 1 : 2;
            bool ok = true;
            int ntile = 0;
            for (int i = 0; i < nu && ok; ++i) {
                const long long u = u0 + i;
                const int c = (int)(u % p.nch), buf = i & 1;
                const bool fresh = i == 0 || c == 0;
                const bool last = c == p.nch - 1 || i == nu - 1;  // the tile's last chunk here
                if (i >= 2 && !(ok = dwait(sm, sm.out_empty[buf], ((i >> 1) - 1) & 1, p.status))) break;
                for (int j = 0; j < NM && ok; ++j) {
                    const int idx = NM * i + j, s = idx % kSlots;
                    if (fresh && !(ok = dwait(sm, sm.a_full[j], ntile & 1, p.status))) break;
                    if (!(ok = dwait(sm, sm.w_full[s], (idx / kSlots) & 1, p.status))) break;
                    tc_fence_after();
                    const uint32_t wb = smem_u32(sm.w[s]);
                    // (straight-line issue: a loop with a run-time trip count around
                    // tcgen05.mma was measured to halve the issue rate)
                    auto issue = [&](int half) {
#pragma unroll
                        for (int kk = 0; kk < 4; ++kk)
                            mma_bf16(tmem + 256 * buf,
                                     smem_desc_sw128(smem_u32(sm.a[j][half]) + kk * 32, 16, 1024),
                                     kOut ? smem_desc_sw128(wb + kk * 2048, 8192, 1024)
                                          : smem_desc_sw128(wb + kk * 32, 16, 1024),
                                     idX, (j > 0 || half > 0 || kk > 0) ? 1u : 0u);
                    };
                    issue(0);
                    if (halves > 1) issue(1);
                    mma_commit(smem_u32(&sm.w_empty[s]));
                    if (last) mma_commit(smem_u32(&sm.a_empty[j]));
                }
                if (!ok) break;
                mma_commit(smem_u32(&sm.out_full[buf]));
                if (fresh) ++ntile;
            }
            if (!ok) {
                // release the epilogue warps
                for (int b2 = 0; b2 < 2; ++b2) mma_commit(smem_u32(&sm.out_full[b2]));
            }
            drain_mmas(smem_u32(&sm.drained));
        }
    } else if (warp >= 4) {
        pdl_trigger();
        const int q = warp & 3, ch = (warp - 4) >> 2;
        const uint32_t lane_off = (uint32_t)(q * 32) << 16;
        uint8_t *xb = sm.stage[warp - 4];
        const int cu = lane & 7;
        int my_row = -1;     // b*T + I of tile row 32 q + lane, -1 past B*k
        float my_dl = 0.f;   // its dlogit (dX)
        for (int i = 0; i < nu; ++i) {
            const long long u = u0 + i;
            const int c = (int)(u % p.nch), buf = i & 1;
            const long long tile = u / p.nch;
            const int h = (int)(tile / p.mt), m0 = (int)(tile % p.mt) * 128;
            if (i == 0 || c == 0) {
                const int m = m0 + q * 32 + lane;
                my_row = m < p.Mtok ? p.gidx[(size_t)h * p.Mtok + m] : -1;
                if (!kOut) my_dl = m < p.Mtok ? p.dlogit[(size_t)h * p.Mtok + m] : 0.f;
            }
            const bool got = dwait(sm, sm.out_full[buf], (i >> 1) & 1, p.status);
            tc_fence_after();
            const bool go = __all_sync(0xffffffffu, got && !*(volatile int *)&sm.abort);
            const uint32_t tb = tmem + 256 * buf + lane_off;
#pragma unroll 1
            for (int s0 = 128 * ch; s0 < 128 * ch + 128; s0 += 32) {
                if (!go) break;
                float v[32];
                tmem_ld32(tb + s0, v);
                stage_f32x32(xb, v, 1.f, lane);
                const int n = c * kChunk + s0 + 4 * cu;
                const bool nin = n < p.d;
                float4 w4 = make_float4(0.f, 0.f, 0.f, 0.f);
                if (!kOut && nin) w4 = *reinterpret_cast<const float4 *>(p.WrT + (size_t)h * p.d + n);
#pragma unroll
                for (int r = 0; r < 8; ++r) {
                    const int rl = (lane >> 3) + 4 * r;
                    const int srow = __shfl_sync(0xffffffffu, my_row, rl);
                    const float dlr = __shfl_sync(0xffffffffu, my_dl, rl);
                    float4 val = *reinterpret_cast<const float4 *>(xb + xoff128(rl, cu));
                    if (srow >= 0 && nin) {
                        if (!kOut) {
                            val.x = fmaf(dlr, w4.x, val.x);
                            val.y = fmaf(dlr, w4.y, val.y);
                            val.z = fmaf(dlr, w4.z, val.z);
                            val.w = fmaf(dlr, w4.w, val.w);
                        }
                        red_add_v4(p.dX + (size_t)srow * p.d + n, val.x, val.y, val.z, val.w);
                    }
                }
                __syncwarp();
            }
            tc_fence_before();
            mbar_arrive(smem_u32(&sm.out_empty[buf]));
            if (!go) break;
        }
    }
    tc_fence_before();
    __syncthreads();
    span_end(p.span);
    if (warp == 2) {
        tc_fence_after();
        tmem_dealloc(tmem, 512);
    }
}

// [H, rows, cols] array of 16-bit elements, box {64, box_rows, 1}.
bool map3(CUtensorMap *m, const void *base, uint64_t H, uint64_t rows, uint64_t cols,
          uint32_t box_rows) {
    const uint64_t dims[3] = {cols, rows, H}, strides[2] = {cols * 2, rows * cols * 2};
    const uint32_t box[3] = {64, box_rows, 1};
    return tmap_bf16(m, base, 3, dims, strides, box);
}

template <bool kOut>
cudaError_t launch_scatter_product(DxParams &p, const Dims &dm, cudaStream_t s) {
    const int Mtok = dm.B * dm.k;
    p.Mtok = Mtok;
    p.d = dm.d;
    p.mt = (Mtok + 127) / 128;
    p.nch = (dm.d + kChunk - 1) / kChunk;
    p.units = (long long)dm.H * p.mt * p.nch;
    p.span = active_span();
    const cudaError_t attr = allow_smem((const void *)scatter_product_kernel<kOut>, kSmem);
    if (attr != cudaSuccess) return attr;
    int dev = 0, sms = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e == cudaSuccess) e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    if (e != cudaSuccess) return e;
    const long long grid = p.units < sms ? p.units : sms;
    e = launch_pdl(scatter_product_kernel<kOut>, dim3((unsigned)grid), dim3(kThreads), kSmem, s, p);
    note_launches(1);
    return e;
}

}  // namespace

cudaError_t tc_dx(const Dims &dm, const void *Wq, const void *Wk, const void *Wv, const Saved &sv,
                  float *dX, cudaStream_t s) {
    DxParams p;
    memset(&p, 0, sizeof(p));
    const int Mtok = dm.B * dm.k;
    if (Mtok <= 0 || dm.d <= 0 || dm.H <= 0) return cudaSuccess;
    p.f16 = dqkv_f16(dm) ? 1 : 0;
    const size_t nw = (size_t)dm.H * dm.d * 64;
    const void *W[3] = {Wq, Wk, Wv};
    if (p.f16)
        for (int j = 0; j < 3; ++j) W[j] = static_cast<const char *>(sv.W16) + 2 * nw * j;
    bool ok = map3(&p.mA, sv.dQKV, dm.H, Mtok, p.f16 ? 256 : 512, 128);
    for (int j = 0; j < 3; ++j) ok = ok && map3(&p.mW[j], W[j], dm.H, dm.d, 64, 256);
    if (!ok) return cudaErrorInvalidValue;
    p.gidx = sv.gidx;
    p.dlogit = sv.dlogit;
    p.WrT = sv.WrT;
    p.dX = dX;
    p.status = sv.status;
    return launch_scatter_product<false>(p, dm, s);
}

cudaError_t tc_out_scatter(const Dims &dm, const void *Wo, const Saved &sv, float *Y,
                           cudaStream_t s) {
    DxParams p;
    memset(&p, 0, sizeof(p));
    const int Mtok = dm.B * dm.k;
    if (Mtok <= 0 || dm.d <= 0 || dm.H <= 0) return cudaSuccess;
    // fp16 attention path: fp16 AR and the fp16 copy of W_o, one MMA per step
    p.f16 = attn_f16(dm) ? 1 : 0;
    const void *wo = p.f16 ? static_cast<const void *>(wo16_of(dm, sv)) : Wo;
    bool ok = p.f16 ? map3(&p.mA, sv.AR16, dm.H, Mtok, 64, 128) : map3(&p.mA, sv.AR, dm.H, Mtok, 128, 128);
    ok = ok && map3(&p.mW[0], wo, dm.H, 64, dm.d, 64);
    if (!ok) return cudaErrorInvalidValue;
    p.gidx = sv.gidx;
    p.dX = Y;
    p.status = sv.status;
    return launch_scatter_product<true>(p, dm, s);
}

}  // namespace mosa
