// Token-major form of the two products that add the heads' rows into a
// [B*T, d] array (Sec. 2.2, Eq. mosa_mha):
//   output F5:          Y[t, n]  = sum_h AR_h(pos_h(t), :) W_o[h](:, n)
//   input gradient B3:  dX[t, n] = sum_h sum_j [dQ|dK|dV]_{h,j}(pos_h(t), :) W_j[h](n, :)
//                                  + sum_h dlogit_h(pos_h(t)) W_r[n, h]
// where pos_h(t) is the row of head h's selected list holding token t (the
// term is absent when head h did not select t).
//
// The row-major form (tc_dx.cu) computes each head's rows and scatter-adds
// them, H-fold fp32 reductions into the output through L2.  When every head
// keeps a large share of the tokens (k >= T/2; every dense or local head of
// a hybrid layer keeps all of them) this form is cheaper for F5: a unit owns a tile of 128 consecutive tokens of one sequence and
// 256 output columns, gathers each head's rows for those tokens (zeros for
// tokens the head did not select) as the A operand, sums all heads' products
// in one TMEM accumulator and writes the tile once, with plain stores and no
// zeroing of the output beforehand.  The tensor cores then also multiply the
// zero rows, T/k times the algorithmic MMA work, which the removed reductions
// more than pay for while T/k is small.
//
// Operands: F5 gathers AR as fp16 rows (one MMA per head and 16-wide K step,
// K = 64; bf16 hi/lo pairs, two MMAs, where the attention runs on the pair
// path) and streams W_o[h] (its fp16 copy, or bf16) as 64 x 256 MN-major
// blocks; dX gathers the fp16 dQ|dK|dV rows
// (one 64-column part per stage, K = 64) and streams the fp16 copies of W_j[h]
// as 256 x 64 K-major blocks; the dlogit term is added in the epilogue from
// the fp32 transpose of W_r.
//
// A persistent grid (at most one CTA per SM) takes contiguous ranges of the
// units (token tile major, column chunk minor); each unit is H (F5) or 3H (dX)
// stages through a 3-slot ring; the accumulators alternate between two
// 256-column halves of TMEM so the epilogue of one unit runs under the MMAs
// of the next.
// Warps: 0 TMA producer (weights), 1 MMA issuer, 2 TMEM owner, 3 idle,
// 4-7 gather the A rows (cp.async, 8 threads per 128-byte row segment),
// 8-11 epilogue (warp w: tile rows 32 (w % 4) .. +31).  Every wait is bounded.
#include <cstdlib>
#include <mutex>

#include "launch.h"
#include "profile.h"
#include "tc_common.cuh"
#include "tc_tiles.cuh"
#include "tmap.h"

namespace mosa {
namespace {

using namespace tc;

constexpr int kHsThreads = 384;
constexpr int kHsMaxSlots = 4;
constexpr int kHsChunk = 256;            // output columns per unit
constexpr int kHsMaxDlHeads = 16;        // dX: heads whose dlogit rows the epilogue stages
constexpr int kWBlock = 32768;           // weight bytes per stage: 64 x 256 (F5) or 256 x 64 (dX)

template <bool kOut>
struct HsCfg {
    static constexpr int A_BYTES = kOut ? 2 * kTileHalf : kTileHalf;   // AR pair, or one fp16 part
    static constexpr int SLOT = A_BYTES + kWBlock;
    static constexpr int P = kOut ? 1 : 3;                               // stages per head
    static constexpr int ROW_BYTES = kOut ? 256 : 512;                   // gathered row in global memory
    static constexpr int SLOTS = kOut ? 3 : 4;                           // ring depth (shared memory)
    static constexpr int LAG = SLOTS - 2;   // gathered stages are confirmed this many stages late
};

template <bool kOut>
struct HsSmem {
    uint8_t ring[HsCfg<kOut>::SLOTS][HsCfg<kOut>::SLOT];
    uint8_t stage[4][4096];                        // epilogue staging, one per epilogue warp
    float dl[kOut ? 1 : 128][kOut ? 1 : kHsMaxDlHeads];   // dX: dlogit_h(pos_h(t)) of the tile rows
    uint64_t full[kHsMaxSlots], empty[kHsMaxSlots], acc_full[2], acc_empty[2], drained;
    uint32_t tmem;
    int abort;
};
template <bool kOut>
constexpr int hs_smem() { return (int)sizeof(HsSmem<kOut>) + 1024; }
static_assert(sizeof(HsSmem<true>) + 1024 <= 227 * 1024, "shared memory");
static_assert(sizeof(HsSmem<false>) + 1024 <= 227 * 1024, "shared memory");

struct HsParams {
    CUtensorMap mW[3];      // F5: W_o [H, 64, d], box {64, 64, 1}; dX: fp16 W_j [H, d, 64], box {64, 256, 1}
    const uint8_t *A;       // F5: AR pairs [H, B*k, 128] bf16; dX: fp16 dQ|dK|dV|dlogit rows [H, B*k, 256]
    const int32_t *pos;     // [H, B*T]: row b*k + i of head h holding token (b, t), or -1
    const float *dlogit;    // dX: [H, B*k]
    const float *WrT;       // dX: [H, d] fp32 transpose of W_r
    float *out;             // [B*T, d]: Y or dX
    int accumulate;         // add to out instead of overwriting it
    int f16;                // F5: A = fp16 AR rows [H, B*k, 64] and W = the fp16 copy of W_o (one MMA)
    int B, T, d, H, Mtok;
    int tps, nch;           // token tiles per sequence, column chunks
    long long units;        // B * tps * nch
    uint32_t *status;
    unsigned long long *span;
};

template <bool kOut>
__device__ __forceinline__ bool hwait(HsSmem<kOut> &sm, uint64_t &bar, uint32_t parity,
                                      uint32_t *status) {
    if (*(volatile int *)&sm.abort) return false;
    if (mbar_wait(smem_u32(&bar), parity)) return true;
    atomicOr(status, kStatusTimeout);
    *(volatile int *)&sm.abort = 1;
    return false;
}

// Unit u -> sequence b, first token t0 of the tile, first column c0.
__device__ __forceinline__ void hs_unit(const HsParams &p, long long u, int &b, int &t0, int &c0) {
    const long long tile = u / p.nch;
    c0 = (int)(u % p.nch) * kHsChunk;
    b = (int)(tile / p.tps);
    t0 = (int)(tile % p.tps) * 128;
}

template <bool kOut>
__global__ void __launch_bounds__(kHsThreads, 1) head_sum_kernel(const __grid_constant__ HsParams p) {
    using C = HsCfg<kOut>;
    extern __shared__ uint8_t smem_raw[];
    HsSmem<kOut> &sm = *reinterpret_cast<HsSmem<kOut> *>(
        (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    // this CTA's units [u0, u1)
    const long long u0 = p.units * blockIdx.x / gridDim.x;
    const long long u1 = p.units * (blockIdx.x + 1) / gridDim.x;
    const int nu = (int)(u1 - u0);
    const int spu = p.H * C::P;   // stages per unit
    const size_t BT = (size_t)p.B * p.T;

    if (threadIdx.x == 0) {
        for (int s = 0; s < C::SLOTS; ++s) {
            mbar_init(smem_u32(&sm.full[s]), 1 + 128);   // the TMA arrival plus one per gatherer
            mbar_init(smem_u32(&sm.empty[s]), 1);
        }
        for (int i = 0; i < 2; ++i) {
            mbar_init(smem_u32(&sm.acc_full[i]), 1);
            mbar_init(smem_u32(&sm.acc_empty[i]), 128);
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
    pdl_wait();  // A rows, pos and dlogit come from earlier kernels
    span_begin(p.span);

    if (warp == 0) {
        // ------------------------------------------------ weight blocks (TMA)
        if (lane == 0) {
            int issued = 0;
            bool ok = true;
            for (int i = 0; i < nu && ok; ++i) {
                int b, t0, c0;
                hs_unit(p, u0 + i, b, t0, c0);
                for (int st = 0; st < spu; ++st) {
                    const int it = i * spu + st, s = it % C::SLOTS;
                    if (!(ok = hwait(sm, sm.empty[s], ((it / C::SLOTS) & 1) ^ 1, p.status))) break;
                    const int h = st / C::P, j = st % C::P;
                    const uint32_t fb = smem_u32(&sm.full[s]);
                    const uint32_t wb = smem_u32(sm.ring[s] + C::A_BYTES);
                    mbar_expect_tx(fb, kWBlock);
                    if (kOut) {
                        // W_o[h] rows 0..63 (K), columns c0 .. c0+255 (N) as four 64-wide blocks
                        for (int q = 0; q < 4; ++q) tma_load_3d(wb + q * 8192, &p.mW[0], fb, c0 + 64 * q, 0, h);
                    } else {
                        // W_j[h] rows c0 .. c0+255 (N), 64 columns (K)
                        tma_load_3d(wb, &p.mW[j], fb, 0, c0, h);
                    }
                    issued = it + 1;
                }
            }
            // drain: the last load of every slot has landed (a stage whose
            // gathering threads gave up before issuing it never completes;
            // its wait then runs out the full bound)
            for (int it = max(0, issued - C::SLOTS); it < issued; ++it)
                drain_phase(smem_u32(&sm.full[it % C::SLOTS]), (it / C::SLOTS) & 1);
        }
    } else if (warp == 1) {
        // ---------------------------------------------------------- MMA issue
        if (lane == 0) {
            const uint32_t idesc = kOut ? (p.f16 ? idesc_f16(128, kHsChunk, false, true)
                                                 : idesc_bf16(128, kHsChunk, false, true))
                                        : idesc_f16(128, kHsChunk, false, false);
            const int halves = p.f16 ? 1 : 2;
            bool ok = true;
            for (int i = 0; i < nu && ok; ++i) {
                const int buf = i & 1;
                // the epilogue has read this accumulator's previous unit
                if (i >= 2 && !(ok = hwait(sm, sm.acc_empty[buf], ((i >> 1) - 1) & 1, p.status))) break;
                tc_fence_after();
                const uint32_t acc = tmem + 256 * buf;
                for (int st = 0; st < spu; ++st) {
                    const int it = i * spu + st, s = it % C::SLOTS;
                    if (!(ok = hwait(sm, sm.full[s], (it / C::SLOTS) & 1, p.status))) break;
                    tc_fence_after();
                    const uint32_t a = smem_u32(sm.ring[s]), wb = a + C::A_BYTES;
                    const uint32_t first = st > 0 ? 1u : 0u;
                    // (straight-line issue: a loop with a run-time trip count around
                    // tcgen05.mma halves the issue rate)
                    if (kOut) {
#pragma unroll
                        for (int kk = 0; kk < 4; ++kk)
                            mma_bf16(acc, smem_desc_sw128(a + kk * 32, 16, 1024),
                                     smem_desc_sw128(wb + kk * 2048, 8192, 1024), idesc,
                                     kk > 0 ? 1u : first);
                        if (halves > 1) {   // the lo half of the AR pair
#pragma unroll
                            for (int kk = 0; kk < 4; ++kk)
                                mma_bf16(acc, smem_desc_sw128(a + kTileHalf + kk * 32, 16, 1024),
                                         smem_desc_sw128(wb + kk * 2048, 8192, 1024), idesc, 1u);
                        }
                    } else {
#pragma unroll
                        for (int kk = 0; kk < 4; ++kk)
                            mma_bf16(acc, smem_desc_sw128(a + kk * 32, 16, 1024),
                                     smem_desc_sw128(wb + kk * 32, 16, 1024), idesc,
                                     kk > 0 ? 1u : first);
                    }
                    mma_commit(smem_u32(&sm.empty[s]));
                }
                if (!ok) break;
                mma_commit(smem_u32(&sm.acc_full[buf]));
            }
            if (!ok) {
                // release the epilogue warps (their later waits see the abort flag)
                for (int b2 = 0; b2 < 2; ++b2) mma_commit(smem_u32(&sm.acc_full[b2]));
            }
            drain_mmas(smem_u32(&sm.drained));
        }
    } else if (warp >= 4 && warp < 8) {
        // ------------------------------------------------- A rows (cp.async)
        // thread t copies 16-byte chunk (t & 7) of tile rows (t >> 3) + 16 j,
        // j = 0..7: each warp instruction covers four whole 128-byte segments
        const int t = threadIdx.x - 128;
        const int chunk = t & 7, sub = t >> 3;
        const int row_bytes = (kOut && p.f16) ? 128 : C::ROW_BYTES;   // fp16 AR rows: 64 values
        int landed = 0, issued = 0;
        bool ok = true;
        // this thread's rows of head h's list for the tile of (unit i, head h),
        // -1 where the head did not select the token; loaded one head ahead
        auto load_rows = [&](int i, int h, int (&pr)[8]) {
            int b, t0, c0;
            hs_unit(p, u0 + i, b, t0, c0);
#pragma unroll
            for (int j = 0; j < 8; ++j) {
                const int tt = t0 + sub + 16 * j;
                pr[j] = tt < p.T ? __ldg(p.pos + (size_t)h * BT + (size_t)b * p.T + tt) : -1;
            }
        };
        int prow[8], pnext[8];
        if (nu > 0) load_rows(0, 0, pnext);
        for (int i = 0; i < nu && ok; ++i) {
            for (int h = 0; h < p.H && ok; ++h) {
#pragma unroll
                for (int j = 0; j < 8; ++j) prow[j] = pnext[j];
                if (h + 1 < p.H)
                    load_rows(i, h + 1, pnext);
                else if (i + 1 < nu)
                    load_rows(i + 1, 0, pnext);
#pragma unroll 1
                for (int part = 0; part < C::P; ++part) {
                    const int it = i * spu + h * C::P + part, s = it % C::SLOTS;
                    if (!(ok = hwait(sm, sm.empty[s], ((it / C::SLOTS) & 1) ^ 1, p.status))) break;
                    const uint32_t a = smem_u32(sm.ring[s]);
#pragma unroll
                    for (int j = 0; j < 8; ++j) {
                        const int r = sub + 16 * j;
                        const int pr = prow[j];
                        const uint32_t nbytes = pr >= 0 ? 16u : 0u;
                        const uint8_t *src = p.A + ((size_t)h * p.Mtok + (pr >= 0 ? pr : 0)) * row_bytes +
                                             part * 128 + chunk * 16;
                        const uint32_t off = r * 128 + ((chunk ^ (r & 7)) << 4);
                        cp_async16(a + off, src, nbytes);
                        if (kOut && !p.f16) cp_async16(a + kTileHalf + off, src + 128, nbytes);   // lo half
                    }
                    cp_async_commit();
                    issued = it + 1;
                    if (it >= C::LAG) {
                        cp_async_wait<C::LAG>();
                        fence_proxy_async();
                        mbar_arrive(smem_u32(&sm.full[(it - C::LAG) % C::SLOTS]));
                        ++landed;
                    }
                }
            }
        }
        // every stage issued lands before its barrier is arrived on, also after a give-up
        cp_async_wait<0>();
        fence_proxy_async();
        for (int it = landed; it < issued; ++it) mbar_arrive(smem_u32(&sm.full[it % C::SLOTS]));
    } else if (warp >= 8) {
        // ------------------------------------------------------------ epilogue
        pdl_trigger();
        const int q = warp & 3;
        const int r = q * 32 + lane;            // tile row of this thread's TMEM lane
        const uint32_t lane_off = (uint32_t)(q * 32) << 16;
        uint8_t *xb = sm.stage[q];
        const int cu = lane & 7;
        for (int i = 0; i < nu; ++i) {
            int b, t0, c0;
            hs_unit(p, u0 + i, b, t0, c0);
            const int buf = i & 1;
            if (!kOut) {
                // dlogit_h(pos_h(t)) of this thread's row, read back by its own warp
                // (all heads' loads in flight together: two round trips)
                const int tt = t0 + r;
                int pr[kHsMaxDlHeads];
#pragma unroll
                for (int h = 0; h < kHsMaxDlHeads; ++h)
                    pr[h] = (h < p.H && tt < p.T) ? __ldg(p.pos + (size_t)h * BT + (size_t)b * p.T + tt) : -1;
#pragma unroll
                for (int h = 0; h < kHsMaxDlHeads; ++h)
                    sm.dl[r][h] = pr[h] >= 0 ? __ldg(p.dlogit + (size_t)h * p.Mtok + pr[h]) : 0.f;
                __syncwarp();
            }
            const bool got = hwait(sm, sm.acc_full[buf], (i >> 1) & 1, p.status);
            tc_fence_after();
            const bool go = __all_sync(0xffffffffu, got && !*(volatile int *)&sm.abort);
            const uint32_t tb = tmem + 256 * buf + lane_off;
#pragma unroll 1
            for (int g = 0; g < kHsChunk / 32 && go; ++g) {
                float v[32];
                tmem_ld32(tb + 32 * g, v);
                stage_f32x32(xb, v, 1.f, lane);   // ends with __syncwarp
                const int col = c0 + 32 * g + 4 * cu;
                float4 val[8];
#pragma unroll
                for (int rr = 0; rr < 8; ++rr)
                    val[rr] = *reinterpret_cast<const float4 *>(xb + xoff128((lane >> 3) + 4 * rr, cu));
                if (!kOut && col < p.d) {
                    for (int h = 0; h < p.H; ++h) {
                        const float4 w = __ldg(reinterpret_cast<const float4 *>(p.WrT + (size_t)h * p.d + col));
#pragma unroll
                        for (int rr = 0; rr < 8; ++rr) {
                            const float dl = sm.dl[q * 32 + (lane >> 3) + 4 * rr][h];
                            val[rr].x = fmaf(dl, w.x, val[rr].x);
                            val[rr].y = fmaf(dl, w.y, val[rr].y);
                            val[rr].z = fmaf(dl, w.z, val[rr].z);
                            val[rr].w = fmaf(dl, w.w, val[rr].w);
                        }
                    }
                }
#pragma unroll
                for (int rr = 0; rr < 8; ++rr) {
                    const int tt = t0 + q * 32 + (lane >> 3) + 4 * rr;
                    if (tt < p.T && col < p.d) {
                        float *dst = p.out + ((size_t)b * p.T + tt) * p.d + col;
                        // adding into the output: one reduction per element (no
                        // round trip), else a plain store
                        if (p.accumulate)
                            red_add_v4(dst, val[rr].x, val[rr].y, val[rr].z, val[rr].w);
                        else
                            *reinterpret_cast<float4 *>(dst) = val[rr];
                    }
                }
                __syncwarp();
            }
            tc_fence_before();
            mbar_arrive(smem_u32(&sm.acc_empty[buf]));
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

// pos[h, b*T + t] = b*k + i where I[b,h,i] = t, else -1: one CTA per (b, h).
// The selected lists are strictly ascending and in range (the selection
// produces them so, and caller-given lists are checked and replaced when they
// are not), so every token appears at most once per head.
__global__ void token_rows_kernel(const int32_t *__restrict__ gidx, int32_t *__restrict__ pos, int B,
                                  int T, int k) {
    const int b = blockIdx.x, h = blockIdx.y;
    int32_t *row = pos + ((size_t)h * B + b) * T;
    for (int t = threadIdx.x; t < T; t += blockDim.x) row[t] = -1;
    __syncthreads();
    const int32_t *g = gidx + ((size_t)h * B + b) * k;
    for (int i = threadIdx.x; i < k; i += blockDim.x) {
        const int t = g[i] - b * T;
        if (t >= 0 && t < T) row[t] = b * k + i;
    }
}

// MOSA_HEADSUM: unset = the measured policy below; 0 = row-major products only;
// 1 = token-major products wherever they apply, whatever T/k (tests).
int headsum_mode() {
    const char *v = std::getenv("MOSA_HEADSUM");
    if (v == nullptr || v[0] == '\0') return -1;
    return v[0] == '0' ? 0 : 1;
}

bool map_w(CUtensorMap *m, const void *base, uint64_t H, uint64_t rows, uint64_t cols, uint32_t box_rows) {
    const uint64_t dims[3] = {cols, rows, H}, strides[2] = {cols * 2, rows * cols * 2};
    const uint32_t box[3] = {64, box_rows, 1};
    return tmap_bf16(m, base, 3, dims, strides, box);
}

template <bool kOut>
cudaError_t launch_head_sum(HsParams &p, const Dims &dm, cudaStream_t s) {
    p.B = dm.B;
    p.T = dm.T;
    p.d = dm.d;
    p.H = dm.H;
    p.Mtok = dm.B * dm.k;
    p.tps = (dm.T + 127) / 128;
    p.nch = (dm.d + kHsChunk - 1) / kHsChunk;
    p.units = (long long)dm.B * p.tps * p.nch;
    p.span = active_span();
    if (p.units <= 0) return cudaSuccess;
    constexpr int smem = hs_smem<kOut>();
    const cudaError_t attr = allow_smem((const void *)head_sum_kernel<kOut>, smem);
    if (attr != cudaSuccess) return attr;
    int dev = 0, sms = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e == cudaSuccess) e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    if (e != cudaSuccess) return e;
    const long long grid = p.units < sms ? p.units : sms;
    e = launch_pdl(head_sum_kernel<kOut>, dim3((unsigned)grid), dim3(kHsThreads), smem, s, p);
    note_launches(1);
    return e;
}

}  // namespace

// Policy (measured at B4 T4096 d1024 with H8 k2048 and H16 k1024): the
// token-major output product beats the scatter-add one at T = 2k (59 -> 41 us)
// and ties at T = 4k, where it does four times the algorithmic MMA work; the
// token-major input gradient, whose per-stage operands (16 KB of gathered
// rows and 32 KB of weights for 0.26 us of MMAs) leave it bound by L2 latency
// times the bytes a 4-slot ring can hold in flight, ran slower than the
// row-major one at T = 2k, so it is used only when forced.
bool use_headsum_out(const Dims &dm) {
    const int mode = headsum_mode();
    if (mode == 0 || !use_tc(dm) || dm.k <= 128 || dm.d % 8 != 0) return false;
    return mode == 1 || (long long)dm.T <= 2LL * dm.k;
}

bool use_headsum_dx(const Dims &dm) {
    const int mode = headsum_mode();
    if (mode != 1 || !attn_f16(dm) || dm.d % 8 != 0 || dm.H > kHsMaxDlHeads) return false;
    return true;
}

cudaError_t tc_token_rows(const Dims &dm, const Saved &sv, cudaStream_t s) {
    if (dm.B <= 0 || dm.H <= 0 || dm.T <= 0) return cudaSuccess;
    token_rows_kernel<<<dim3(dm.B, dm.H), 256, 0, s>>>(sv.gidx, sv.pos, dm.B, dm.T, dm.k);
    note_launches(1);
    return cudaGetLastError();
}

cudaError_t tc_out_headsum(const Dims &dm, const void *Wo, const Saved &sv, float *Y, cudaStream_t s) {
    HsParams p;
    memset(&p, 0, sizeof(p));
    // fp16 attention path (k > 128, always so here): fp16 AR and the fp16 copy
    // of W_o that the forward made beside TopK, one MMA per step
    p.f16 = attn_f16(dm) ? 1 : 0;
    const void *wo = p.f16 ? static_cast<const void *>(wo16_of(dm, sv)) : Wo;
    if (!map_w(&p.mW[0], wo, dm.H, 64, dm.d, 64)) return cudaErrorInvalidValue;
    p.A = static_cast<const uint8_t *>(p.f16 ? sv.AR16 : sv.AR);
    p.pos = sv.pos;
    p.out = Y;
    p.accumulate = dm.accumulate ? 1 : 0;
    p.status = sv.status;
    return launch_head_sum<true>(p, dm, s);
}

cudaError_t tc_dx_headsum(const Dims &dm, const Saved &sv, float *dX, cudaStream_t s) {
    HsParams p;
    memset(&p, 0, sizeof(p));
    const size_t nw = (size_t)dm.H * dm.d * 64;
    for (int j = 0; j < 3; ++j)
        if (!map_w(&p.mW[j], static_cast<const char *>(sv.W16) + 2 * nw * j, dm.H, dm.d, 64, 256))
            return cudaErrorInvalidValue;
    p.A = static_cast<const uint8_t *>(sv.dQKV);
    p.pos = sv.pos;
    p.dlogit = sv.dlogit;
    p.WrT = sv.WrT;
    p.out = dX;
    p.accumulate = dm.accumulate ? 1 : 0;
    p.status = sv.status;
    return launch_head_sum<false>(p, dm, s);
}

}  // namespace mosa
