// Index-masked causal attention over the k selected tokens of each head on
// the tcgen05 tensor cores (Sec. 2.1 Eq. attention with the MoSA mask of
// Sec. 2.2; with I strictly ascending, I_i >= I_j is j <= i).
//
// Forward (F4), one CTA per (128-query tile, sequence b, head h):
//   for each 128-key block j (causal: up to the tile's last query)
//     S_j  = Q K_j^T                       tcgen05, fp32 in TMEM, two buffers
//     P_j  = exp(S_j/sqrt(h') - m), running max m and sum l per row
//     O   += P_j V_j                       tcgen05, O in TMEM; P read from TMEM
//                                          (k > 128) or shared memory (k <= 128)
//   A = O / l, AR = r A, lse = m + log l  (details at the kernel).
// Precision.  For k <= 128, Q, K, V, P, dA and dS are bf16 hi/lo pairs
// (v ~ hi + lo), so each product is three bf16 MMAs (hi*hi + hi*lo + lo*hi)
// into one fp32 accumulator, at fp32-level accuracy.  For k > 128 they are
// single fp16 values (11-bit significand, 8 times finer than bf16) and each
// product is one MMA; the operands that meet the bf16 weights outside the
// attention (diag(r) A and dQ|dK|dV) stay pairs either way.  A measured
// audit of the rounding of each intermediate against the stated tolerances
// chose this split; an fp16 value at or beyond the fp16 range sets
// kStatusRange instead of passing silently.
// Backward (B2), flash-style with P recomputed from the saved log-sum-exp,
// D = rowsum(dA o A) and dS = P o (dP - D): one CTA per (128-key tile, b, h)
// over 128-query blocks: S = Q K^T, dP = dA V^T, then dV += P^T dA,
// dK += dS^T Q, and dQ = dS K added into an fp32 accumulator (details at the
// kernel); k <= 128 needs one block and writes dQ directly.
// The same shared-memory tile of Q (or dA, K) serves as a K-major operand in
// one product and as an MN-major operand in the other.
// Warp roles: 0 TMA producer, 1 MMA issuer, 2 TMEM allocator, 4-11 softmax
// and epilogue warps, two threads per row (each half of the keys).  All waits
// are bounded.
#include <mutex>

#include "launch.h"
#include "profile.h"
#include "tc_common.cuh"
#include "tc_tiles.cuh"
#include "tmap.h"

namespace mosa {
namespace {

using namespace tc;

constexpr int kQ = 128;          // queries per CTA

struct AttnParams {
    CUtensorMap mQ, mK, mV;   // 4-D maps over [H, B, k, 128] pairs, box {64, rows, 1, 1}
                              // (k <= 128: 3-D maps over [H, B*k, 128], box {64, 128, 1})
    int k, B, Mtok;
    int U;                    // k <= 128: sequences packed into one 128-row tile
    float scale_log2;         // log2(e) / sqrt(h')
    const float *rsel;        // [H, B*k]
    bf16 *AR;                 // [H, B*k, 128] pair
    __half *AR16;             // k > 128: [H, B*k, 64] fp16 AR as well (the output product's operand)
    float *lse;               // [H, B*k]
    uint32_t *status;
    unsigned long long *span; // measurement: kernel span slot, or null
};


// Forward for k > 128 (F4), one CTA per (128-query tile, b, h), 384 threads:
// warps 0-3 load, issue MMAs and own TMEM; warps 4-11 run the softmax, two per
// TMEM lane quadrant (warp w: query rows 32 (w % 4) .. +31, keys
// 64 ((w - 4) / 4) .. +63 of each 128-key block).  Q, K, V and P are fp16
// (one MMA per 16-wide K step).  For key block j:
//   S_j = Q K_j^T into TMEM buffer j % 2;
//   P_j = exp2(S_j scale - m) with m the row's running maximum, updated only
//   when the block's maximum exceeds it by more than 2^8 (O and l are then
//   rescaled in place; otherwise P may reach 2^8, well inside the fp16 range,
//   and the final O / l uses the same m throughout), written as fp16 into
//   TMEM buffer j % 2 (two fp16 per 32-bit column, 64 columns);
//   O += P_j V_j with P read from TMEM as the A operand and V from shared
//   memory, O in TMEM.
// P in TMEM takes the shared-memory stores and the proxy fence of P off the
// softmax warps' chain (47.7 -> 44.6 us at B4 T4096 d1024 H8 k2048); the
// MMAs themselves cost the same either way (measured with %clock stamps:
// about 120 cycles per M = 128, N = 64, K = 16 instruction and 165 at
// N = 128, also when independent accumulators alternate, so the tensor pipe
// runs these small instructions one after another at a fixed cost each).
// Earlier builds found that a tcgen05.st issued while an MMA reads its A
// operand from TMEM corrupts that MMA even when the columns differ, so the
// softmax warps store P_j only after P_{j-1} V_{j-1} has completed (issued a
// whole softmax earlier, so the wait is normally over at once) and no other
// TMEM store (the rescale of O) happens while one runs.
// The MMA issuer issues S_{j+2} as soon as the softmax warps have read S_j
// into registers and P_j V_j as soon as P_j is stored, so the softmax of one
// block runs while the MMAs of the neighbouring blocks do.  Each hand-over
// barrier comes in a pair, one per buffer parity, so no waiter can see its
// barrier complete twice ahead of it.
// K and V blocks stream through an 8-slot ring in the order the MMAs use
// them: K0, K1, K2, V0, K3, V1, ... (see kv_item).
constexpr int kLT = 384;              // threads
constexpr int kLWorkers = 256;
constexpr int kLKeys = 128;           // keys per block
constexpr int kLSlots = 8;            // ring slots of one K or V block (16 KB)
constexpr float kRescaleLog2 = 8.f;   // lazy-rescale threshold (log2 units)

struct FwdLargeSmem {
    uint8_t q[kTileHalf];                     // Q, fp16 [128 x 64]
    uint8_t kv[kLSlots][kTileHalf];           // K or V blocks, fp16 [128 x 64]
    float part[2][2][128];                    // [block parity][key half]: block max, final sums
    uint64_t q_full, kv_full[kLSlots], kv_empty[kLSlots];
    uint64_t s_full[2], s_free[2], p_ready[2], pv_done[2];   // per buffer parity
    uint64_t drained;                                         // the MMA issuer's final drain
    uint32_t tmem;
    int abort;
};
constexpr int kFwdLargeSmem = (int)sizeof(FwdLargeSmem) + 1024;
static_assert(kFwdLargeSmem <= 227 * 1024, "shared memory");

// Item t of the K/V stream for n blocks, in MMA issue order: K_0, K_1, then
// K_{j+2} followed by V_j while j + 2 < n, then the remaining V_j.
// Returns (is V, block).
__device__ __forceinline__ void kv_item(int t, int n, bool &is_v, int &blk) {
    const int s0 = n < 2 ? n : 2;
    if (t < s0) { is_v = false; blk = t; return; }
    const int u = t - s0, pairs = n > 2 ? n - 2 : 0;
    if (u < 2 * pairs) {
        is_v = (u & 1) == 1;
        blk = is_v ? (u >> 1) : (u >> 1) + 2;
        return;
    }
    is_v = true;
    blk = pairs + (u - 2 * pairs);
}

__device__ __forceinline__ bool lwait(FwdLargeSmem &sm, uint64_t &bar, uint32_t parity, uint32_t *status) {
    if (*(volatile int *)&sm.abort) return false;
    if (mbar_wait(smem_u32(&bar), parity)) return true;
    atomicOr(status, kStatusTimeout);
    *(volatile int *)&sm.abort = 1;
    return false;
}

__global__ void __launch_bounds__(kLT, 1) attn_fwd_tc_kernel(const __grid_constant__ AttnParams p) {
    extern __shared__ uint8_t smem_raw[];
    FwdLargeSmem &sm = *reinterpret_cast<FwdLargeSmem *>(
        (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    // heaviest (last) query tiles first: they visit the most key blocks; the
    // tile index is the grid's slowest dimension, so CTAs start in that order
    const int nqt = gridDim.z;
    const int qt = nqt - 1 - (int)blockIdx.z, b = blockIdx.x, h = blockIdx.y;
    const int i0 = qt * kQ;
    const int n = qt + 1;                      // causal: key blocks 0 .. qt
    const int nitems = 2 * n;

    if (threadIdx.x == 0) {
        mbar_init(smem_u32(&sm.q_full), 1);
        for (int s = 0; s < kLSlots; ++s) {
            mbar_init(smem_u32(&sm.kv_full[s]), 1);
            mbar_init(smem_u32(&sm.kv_empty[s]), 1);
        }
        for (int u = 0; u < 2; ++u) {
            mbar_init(smem_u32(&sm.s_full[u]), 1);
            mbar_init(smem_u32(&sm.s_free[u]), kLWorkers);
            mbar_init(smem_u32(&sm.p_ready[u]), kLWorkers);
            mbar_init(smem_u32(&sm.pv_done[u]), 1);
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
    pdl_wait();  // Q, K, V written by the previous kernels
    span_begin(p.span);
    const uint32_t tmem = sm.tmem;
    // S buffers at columns 0 and 128, O at 256, the fp16 P buffers at 320 and 384
    const uint32_t tO = tmem + 256, tP = tmem + 320;

    if (warp == 0) {
        if (lane == 0) {
            const uint32_t qb = smem_u32(&sm.q_full);
            mbar_expect_tx(qb, kTileHalf);
            tma_load_4d(smem_u32(sm.q), &p.mQ, qb, 0, i0, b, h);
            int issued = 0;
            for (int t = 0; t < nitems; ++t) {
                const int s = t % kLSlots;
                if (!lwait(sm, sm.kv_empty[s], ((t / kLSlots) & 1) ^ 1, p.status)) break;
                bool is_v;
                int blk;
                kv_item(t, n, is_v, blk);
                const uint32_t fb = smem_u32(&sm.kv_full[s]);
                mbar_expect_tx(fb, kTileHalf);
                tma_load_4d(smem_u32(sm.kv[s]), is_v ? &p.mV : &p.mK, fb, 0, blk * kLKeys, b, h);
                issued = t + 1;
            }
            // drain: Q and the last load of every slot have landed
            drain_phase(qb, 0);
            for (int t = max(0, issued - kLSlots); t < issued; ++t)
                drain_phase(smem_u32(&sm.kv_full[t % kLSlots]), (t / kLSlots) & 1);
        }
    } else if (warp == 1) {
        if (lane == 0) {
            constexpr uint32_t idS = idesc_f16(128, kLKeys, false, false);
            constexpr uint32_t idO = idesc_f16(128, 64, false, true);
            int t = 0;   // next K/V item to consume
            bool ok = lwait(sm, sm.q_full, 0, p.status);
            auto take = [&]() -> int {   // wait for item t, return its slot
                const int s = t % kLSlots;
                ok = ok && lwait(sm, sm.kv_full[s], (t / kLSlots) & 1, p.status);
                ++t;
                return s;
            };
            auto issue_s = [&](int j) {  // S_j = Q K_j^T into buffer j % 2
                const int s = take();
                if (!ok) return;
                tc_fence_after();
                mma_k64_f16(tmem + 128 * (j & 1), smem_u32(sm.q), smem_u32(sm.kv[s]), idS);
                mma_commit(smem_u32(&sm.s_full[j & 1]));
                mma_commit(smem_u32(&sm.kv_empty[s]));
            };
            issue_s(0);
            if (n > 1) issue_s(1);
            for (int j = 0; j < n && ok; ++j) {
                const int u = j & 1;
                if (j + 2 < n) {
                    // S_{j+2} reuses buffer j % 2 once the workers hold S_j
                    ok = lwait(sm, sm.s_free[u], (j >> 1) & 1, p.status);
                    tc_fence_after();
                    issue_s(j + 2);
                }
                ok = ok && lwait(sm, sm.p_ready[u], (j >> 1) & 1, p.status);
                const int s = take();   // V_j
                if (!ok) break;
                tc_fence_after();
                // O += P_j V_j: P from TMEM buffer j % 2 (8 columns per 16 keys), V MN-major
                const uint32_t vb = smem_u32(sm.kv[s]);
#pragma unroll
                for (int kk = 0; kk < 8; ++kk)
                    mma_bf16_ts(tO, tP + 64 * u + 8 * kk, smem_desc_sw128(vb + kk * 2048, kTileHalf, 1024),
                                idO, (j > 0 || kk > 0) ? 1u : 0u);
                mma_commit(smem_u32(&sm.pv_done[u]));
                mma_commit(smem_u32(&sm.kv_empty[s]));
            }
            if (!ok) {
                // release the softmax warps (their later waits see the abort flag)
                for (int u = 0; u < 2; ++u) {
                    mma_commit(smem_u32(&sm.s_full[u]));
                    mma_commit(smem_u32(&sm.pv_done[u]));
                }
            }
            drain_mmas(smem_u32(&sm.drained));
        }
    } else if (warp >= 4) {
        pdl_trigger();
        const int q = warp & 3, ch = (warp - 4) >> 2;
        const int r = q * 32 + lane;               // query row of the tile
        const int i = i0 + r;
        const uint32_t lane_off = (uint32_t)(q * 32) << 16;
        float m = -INFINITY, l = 0.f;              // running max (log2 units), partial sum
        bool ok = true;
        for (int j = 0; j < n; ++j) {
            const int u = j & 1;
            ok = lwait(sm, sm.s_full[u], (j >> 1) & 1, p.status) && ok;
            tc_fence_after();
            float s[64];
            tmem_ld64(tmem + 128 * u + lane_off + 64 * ch, s);
            tc_fence_before();
            mbar_arrive(smem_u32(&sm.s_free[u]));   // S_{j+2} may overwrite these columns
            if (j == qt) {
                // diagonal block (earlier blocks are wholly visible): key
                // j*128 + 64 ch + c is visible from query i iff c <= lim
                const int lim = i - (j * kLKeys + 64 * ch);
#pragma unroll
                for (int c = 0; c < 64; ++c)
                    if (c > lim) s[c] = -INFINITY;
            }
            // maxima and sums in four independent chains
            float mx[4] = {-INFINITY, -INFINITY, -INFINITY, -INFINITY};
#pragma unroll
            for (int c = 0; c < 64; ++c) mx[c & 3] = fmaxf(mx[c & 3], s[c]);
            float mb = fmaxf(fmaxf(mx[0], mx[1]), fmaxf(mx[2], mx[3])) * p.scale_log2;
            // the exchange buffer alternates with the block parity: the buffer
            // written here was last read before both warps of the row passed
            // the previous block's barrier, so one barrier per block suffices;
            // only the two warps sharing the lane quadrant q synchronise
            sm.part[u][ch][r] = mb;
            named_barrier(1 + q, 64);
            mb = fmaxf(sm.part[u][0][r], sm.part[u][1][r]);
            const bool grow = mb > m + kRescaleLog2;   // same decision in both threads of the row
            const float m_new = grow ? mb : m;
            const float corr = grow ? exp2_fast(m - m_new) : 1.f;   // 0 on the first block
            float sm4[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
            for (int c = 0; c < 64; ++c) {
                s[c] = exp2_fast(fmaf(s[c], p.scale_log2, -m_new));
                sm4[c & 3] += s[c];
            }
            l = l * corr + ((sm4[0] + sm4[1]) + (sm4[2] + sm4[3]));
            m = m_new;
            if (j > 0 && __any_sync(0xffffffffu, grow)) {
                // O holds P_0 V_0 .. P_{j-1} V_{j-1}: all of them done first
                ok = lwait(sm, sm.pv_done[u ^ 1], ((j - 1) >> 1) & 1, p.status) && ok;
                tc_fence_after();
                float o[32];
                tmem_ld32(tO + lane_off + 32 * ch, o);
#pragma unroll
                for (int c = 0; c < 32; ++c) o[c] *= corr;
                tmem_st32(tO + lane_off + 32 * ch, o);
            }
            // no MMA may read TMEM while P_j is stored: P_{j-1} V_{j-1} (and
            // with it every earlier one) has completed
            if (j >= 1) {
                ok = lwait(sm, sm.pv_done[u ^ 1], ((j - 1) >> 1) & 1, p.status) && ok;
                tc_fence_after();
            }
            {
                uint32_t w[32];
#pragma unroll
                for (int c = 0; c < 32; ++c) w[c] = pack_f16x2(s[2 * c], s[2 * c + 1]);
                tmem_st32u(tP + 64 * u + lane_off + 32 * ch, w);   // keys 64 ch .. +63
            }
            tc_fence_before();
            mbar_arrive(smem_u32(&sm.p_ready[u]));
        }
        ok = lwait(sm, sm.pv_done[(n - 1) & 1], ((n - 1) >> 1) & 1, p.status) && ok;
        tc_fence_after();
        sm.part[n & 1][ch][r] = l;
        named_barrier(1 + q, 64);
        l = sm.part[n & 1][0][r] + sm.part[n & 1][1][r];
        float o[32];
        tmem_ld32(tO + lane_off + 32 * ch, o);      // output columns 32 ch .. +31
        const bool live = __all_sync(0xffffffffu, ok && !*(volatile int *)&sm.abort);
        const bool valid = i < p.k;
        const unsigned vmask = __ballot_sync(0xffffffffu, valid);
        const size_t row0 = (size_t)h * p.Mtok + (size_t)b * p.k + i0 + q * 32;
        if (live) {
            uint8_t *xb = &sm.kv[0][0] + (warp - 4) * 4096;   // the ring is idle now
            const float inv = valid ? 1.f / l : 0.f;
            const float rr = valid ? p.rsel[row0 + lane] : 0.f;
            stage_pair32(xb, o, inv * rr, lane);
            store_rows128(xb, lane, [&](int rl, int c) -> uint4 * {
                if (!((vmask >> rl) & 1u)) return nullptr;
                bf16 *base = p.AR + (row0 + rl) * 128 + 32 * ch;
                return c < 4 ? reinterpret_cast<uint4 *>(base) + c
                             : reinterpret_cast<uint4 *>(base + 64) + (c - 4);
            });
            if (p.AR16 != nullptr && valid) {
                // the same 32 values as one fp16 run (64 bytes) of the fp16 AR row
                uint4 *dst = reinterpret_cast<uint4 *>(p.AR16 + (row0 + lane) * 64 + 32 * ch);
                float amax = 0.f;
#pragma unroll
                for (int u = 0; u < 4; ++u) {
                    uint32_t w[4];
#pragma unroll
                    for (int e = 0; e < 4; ++e) {
                        const float a = o[8 * u + 2 * e] * (inv * rr), c = o[8 * u + 2 * e + 1] * (inv * rr);
                        amax = fmaxf(amax, fmaxf(fabsf(a), fabsf(c)));
                        w[e] = pack_f16x2(a, c);
                    }
                    dst[u] = make_uint4(w[0], w[1], w[2], w[3]);
                }
                if (!(amax < kF16Overflow)) atomicOr(p.status, kStatusRange);
            }
            // lse in natural-log units of the scaled scores
            if (ch == 0 && valid) p.lse[row0 + lane] = (m + log2f(l)) * 0.69314718055994531f;
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

// ------------------------------------------------------------ backward

struct BwdParams {
    CUtensorMap mA0, mA1, mB0, mB1;   // dK/dV: K, V (128 rows), Q, dA (64 rows); dQ: Q, dA (128), K, V (64)
                                      // k <= 128: Q, K, V, dA as 3-D maps over [H, B*k, 128]
    CUtensorMap mOut;                 // k <= 128: dQKV [H, B*k, 512], box {64, U k, 1} (stores)
    CUtensorMap mDQ;                  // k > 128: dQ accumulator [H, B, k, 64] fp32, box {32, 32, 1, 1}
                                      // (reductions)
    int k, Mtok;
    int U, B;                         // k <= 128: sequences per tile, batch
    float scale, scale_log2;
    const float *lse, *Dd;            // [H, B*k]
    bf16 *dQKV;                       // k <= 128: [H, B*k, 512] pair: dQ|dK|dV|dlogit hi, then lo
                                      // k > 128: [H, B*k, 256] fp16 dQ|dK|dV|dlogit
    float *dQacc;                     // k > 128: [H, B*k, 64] fp32 dQ accumulator (zeroed)
    uint32_t *status;
    // k > 128 with RoPE: dK is turned back (Sec. 2.2) before its fp16 rounding
    const int32_t *gidx;              // [H, B*k]: b*T + t
    int rope, T;
    RopeTable rope_tab;
    unsigned long long *span; // measurement: kernel span slot, or null
    // k > 128: an fp32 array of zero_n4 float4 (the layer's dX, which the
    // input-gradient product then adds into) that the otherwise idle warp 3
    // of every CTA zeroes, one slice per CTA, while the attention runs
    float4 *zero;
    long long zero_n4;
    // k <= 128: dQ|dK|dV out as single fp16 into [H, B*k, 256] rows (dQ and
    // dK turned back by RoPE first when asked), else as bf16 pairs
    int out16;
};

template <class SM>
__device__ __forceinline__ void flag_timeout_b(SM &sm, uint32_t *status) {
    atomicOr(status, kStatusTimeout);
    *(volatile int *)&sm.abort = 1;
}



// Backward for k > 128 (B2), one CTA per (128-key tile, b, h), 384 threads:
// warps 0-3 load, issue MMAs and own TMEM; warps 4-11 compute P and dS, two
// per TMEM lane quadrant (warp w: query rows 32 (w % 4) .. +31 of the current
// block, keys 64 ((w - 4) / 4) .. +63 of the tile).  Q, K, V, dA, P and dS
// are fp16 (one MMA per 16-wide K step).  For each 128-query block i at or
// after the tile (causal):
//   S = Q_i K^T, dP = dA_i V^T                  (TMEM)
//   P = exp(S / sqrt(h') - lse_i)               (P tile; kept in registers)
//   dV += P^T dA_i                              (TMEM, the tile read MN-major)
//   dS = P o (dP - D_i)                         (dS tile i % 2)
//   dK += dS^T Q_i, dQ_i = dS K                 (TMEM; dQ in buffer i % 2)
//   dQ_i / sqrt(h') is added into an fp32 accumulator [H, B*k, 64] two
//   blocks later: each worker warp stages its 32 x 32 part in the dS tile it
//   is about to overwrite and one lane hands it to the TMA engine as a bulk
//   reduce-add (the 256 threads' own scattered vector reductions took about
//   1 us per block).
// Measured on this GPU, an MMA instruction (M = 128, K = 16) takes about the
// same time for any N up to 128 (about 2.3x longer per FLOP at N = 64 than
// at N = 256), so the 32 MMAs of a block (S, dP: N = 128; dV, dK, dQ: N = 64)
// cost about 4000 cycles and the kernel is bound by keeping the tensor pipe
// issuing.  The MMA issuer therefore waits only for what each product needs:
// S_{i+1} is issued as soon as the workers have read S_i into registers, and
// dP_{i+1}, dK_i and dQ_i as soon as dS_i is stored; the workers do not wait
// for the tensor pipe either: dS and dQ are double-buffered (the smem dS tile
// and the TMEM dQ accumulator of block i are reused by block i + 2, whose dQ
// the workers drain two blocks late), and lse and D of block i+1 are loaded
// during block i.  Barriers of double-buffered data come in pairs, one per
// buffer, so no waiter can see its barrier complete two phases ahead.
// dK / sqrt(h') and dV are written once at the end as fp16 (dK turned back
// by RoPE first when asked) into dQ|dK|dV|dlogit rows.  Q_i and
// dA_i go to ring slots 2 (i % 3) and 2 (i % 3) + 1, so each load is issued
// up to three blocks ahead of its use (a two-block ring left the MMA issuer
// waiting about 1 us per block for Q_{i+1}).
constexpr int kBT = 384;
constexpr int kBWorkers = 256;
constexpr int kBDepth = 3;                 // blocks in the Q / dA ring
constexpr int kBSlots = 2 * kBDepth;

struct BwdLargeSmem {
    uint8_t k[kTileHalf];                  // K tile, fp16 [128 keys x 64]
    uint8_t v[kTileHalf];                  // V tile
    uint8_t ring[kBSlots][kTileHalf];      // Q_i, dA_i (fp16 [128 queries x 64])
    uint8_t p[2][kTileHalf];               // P [128 queries x 128 keys] as two 64-key blocks
    uint8_t ds[2][2][kTileHalf];           // dS of blocks i % 2, the same layout
    uint64_t kv_full, ring_full[kBSlots], ring_empty[kBSlots];
    uint64_t sp_full, dp_full, s_free, p_ready, pv_done, ds_ready, dq_full[2], dq_empty[2], acc_done;
    uint32_t tmem;
    int abort;
};
constexpr int kBwdLargeSmem = (int)sizeof(BwdLargeSmem) + 1024;
static_assert(kBwdLargeSmem <= 227 * 1024, "shared memory");

__device__ __forceinline__ bool bwait(BwdLargeSmem &sm, uint64_t &bar, uint32_t parity, uint32_t *status) {
    if (*(volatile int *)&sm.abort) return false;
    if (mbar_wait(smem_u32(&bar), parity)) return true;
    atomicOr(status, kStatusTimeout);
    *(volatile int *)&sm.abort = 1;
    return false;
}

__global__ void __launch_bounds__(kBT, 1) attn_bwd_tc_kernel(const __grid_constant__ BwdParams p) {
    extern __shared__ uint8_t smem_raw[];
    BwdLargeSmem &sm = *reinterpret_cast<BwdLargeSmem *>(
        (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    // key tile 0 visits the most query blocks; the tile index is the grid's
    // slowest dimension, so CTAs start heaviest first
    const int jt = blockIdx.z, b = blockIdx.x, h = blockIdx.y;
    const int j0 = jt * 128;
    const int nqb = (p.k + 127) / 128;
    const int nb = nqb - jt;                  // query blocks jt .. nqb-1
    const size_t base = (size_t)h * p.Mtok + (size_t)b * p.k;

    if (threadIdx.x == 0) {
        mbar_init(smem_u32(&sm.kv_full), 1);
        for (int s = 0; s < kBSlots; ++s) {
            mbar_init(smem_u32(&sm.ring_full[s]), 1);
            mbar_init(smem_u32(&sm.ring_empty[s]), 1);
        }
        mbar_init(smem_u32(&sm.sp_full), 1);
        mbar_init(smem_u32(&sm.dp_full), 1);
        mbar_init(smem_u32(&sm.s_free), kBWorkers);
        mbar_init(smem_u32(&sm.p_ready), kBWorkers);
        mbar_init(smem_u32(&sm.pv_done), 1);
        mbar_init(smem_u32(&sm.ds_ready), kBWorkers);
        for (int u = 0; u < 2; ++u) {
            mbar_init(smem_u32(&sm.dq_full[u]), 1);
            mbar_init(smem_u32(&sm.dq_empty[u]), kBWorkers);
        }
        mbar_init(smem_u32(&sm.acc_done), 1);
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
    pdl_wait();  // Q, K, V, dA, lse, D written by the previous kernels
    span_begin(p.span);
    const uint32_t tmem = sm.tmem;
    // S, dP, dV, dK, and the two dQ buffers: all 512 columns
    const uint32_t tS = tmem, tDP = tmem + 128, tDV = tmem + 256, tDK = tmem + 320, tDQ = tmem + 384;

    if (warp == 0) {
        if (lane == 0) {
            const uint32_t kb = smem_u32(&sm.kv_full);
            mbar_expect_tx(kb, 2 * kTileHalf);
            tma_load_4d(smem_u32(sm.k), &p.mA0, kb, 0, j0, b, h);
            tma_load_4d(smem_u32(sm.v), &p.mA1, kb, 0, j0, b, h);
            int issued = 0;
            for (int t = 0; t < 2 * nb; ++t) {
                const int i = t >> 1, is_da = t & 1;
                const int s = 2 * (i % kBDepth) + is_da;
                const int use = i / kBDepth;   // earlier loads into this slot
                if (!bwait(sm, sm.ring_empty[s], (use & 1) ^ 1, p.status)) break;
                const int q0 = (jt + i) * 128;
                const uint32_t fb = smem_u32(&sm.ring_full[s]);
                mbar_expect_tx(fb, kTileHalf);
                tma_load_4d(smem_u32(sm.ring[s]), is_da ? &p.mB1 : &p.mB0, fb, 0, q0, b, h);   // dA_i : Q_i
                issued = t + 1;
            }
            // drain: K, V and the last load of every slot (any kBSlots
            // consecutive loads use every slot once) have landed
            drain_phase(kb, 0);
            for (int t = max(0, issued - kBSlots); t < issued; ++t) {
                const int i = t >> 1;
                drain_phase(smem_u32(&sm.ring_full[2 * (i % kBDepth) + (t & 1)]), (i / kBDepth) & 1);
            }
        }
    } else if (warp == 1) {
        if (lane == 0) {
            constexpr uint32_t idKK = idesc_f16(128, 128, false, false);  // S, dP
            constexpr uint32_t idMN = idesc_f16(128, 64, true, true);     // dV, dK
            constexpr uint32_t idKM = idesc_f16(128, 64, false, true);    // dQ
            bool ok = bwait(sm, sm.kv_full, 0, p.status);
            const uint32_t kt = smem_u32(sm.k), vt = smem_u32(sm.v);
            const uint32_t p0 = smem_u32(sm.p[0]);
            // S_i = Q_i K^T (Q_i in slot 2 (i % 3)), dP_i = dA_i V^T (dA_i in the next slot)
            auto issue_s = [&](int i) {
                const int s = 2 * (i % kBDepth);
                ok = ok && bwait(sm, sm.ring_full[s], (i / kBDepth) & 1, p.status);
                if (!ok) return;
                tc_fence_after();
                mma_k64_f16(tS, smem_u32(sm.ring[s]), kt, idKK);
                mma_commit(smem_u32(&sm.sp_full));
            };
            auto issue_dp = [&](int i) {
                const int s = 2 * (i % kBDepth) + 1;
                ok = ok && bwait(sm, sm.ring_full[s], (i / kBDepth) & 1, p.status);
                if (!ok) return;
                tc_fence_after();
                mma_k64_f16(tDP, smem_u32(sm.ring[s]), vt, idKK);
                mma_commit(smem_u32(&sm.dp_full));
            };
            issue_s(0);
            issue_dp(0);
            // Issue order per block follows the workers' progress: S_{i+1} once
            // S_i is in their registers, dV_i once P_i is stored, then dP_{i+1},
            // dK_i and dQ_i once dS_i is stored (by then dP_i has been read;
            // dQ_i also waits for dQ_{i-2}, the last user of its buffer, to be
            // drained).
            for (int i = 0; i < nb && ok; ++i) {
                const int sq = 2 * (i % kBDepth), sa = sq + 1;
                if (i + 1 < nb) {
                    if (!(ok = bwait(sm, sm.s_free, i & 1, p.status))) break;
                    issue_s(i + 1);
                }
                if (!(ok = ok && bwait(sm, sm.p_ready, i & 1, p.status))) break;
                tc_fence_after();
                mma_k128_f16(tDV, p0, smem_u32(sm.ring[sa]), true, idMN, i > 0);   // dV += P^T dA_i
                mma_commit(smem_u32(&sm.pv_done));                                // P tile free
                mma_commit(smem_u32(&sm.ring_empty[sa]));                         // dA_i (dP_i done too)
                if (!(ok = ok && bwait(sm, sm.ds_ready, i & 1, p.status))) break;
                if (i + 1 < nb) issue_dp(i + 1);
                // dQ_{i-2} drained (the (i/2 - 1)-th completion of buffer i % 2's barrier)
                if (i >= 2) ok = ok && bwait(sm, sm.dq_empty[i & 1], ((i >> 1) - 1) & 1, p.status);
                if (!ok) break;
                tc_fence_after();
                const uint32_t dsb = smem_u32(sm.ds[i & 1][0]);
                mma_k128_f16(tDK, dsb, smem_u32(sm.ring[sq]), true, idMN, i > 0);   // dK += dS^T Q_i
                mma_k128_f16(tDQ + 64 * (i & 1), dsb, kt, false, idKM, false);      // dQ_i = dS K
                mma_commit(smem_u32(&sm.dq_full[i & 1]));
                mma_commit(smem_u32(&sm.ring_empty[sq]));
            }
            if (!ok) {
                // release every wait of the workers that may still be pending
                // (each of their later waits then sees the abort flag first)
                mma_commit(smem_u32(&sm.sp_full));
                mma_commit(smem_u32(&sm.dp_full));
                mma_commit(smem_u32(&sm.pv_done));
                mma_commit(smem_u32(&sm.dq_full[0]));
                mma_commit(smem_u32(&sm.dq_full[1]));
            }
            // acc_done's only phase covers every MMA issued: wait for it here too
            // (the workers' own wait gives up at once when the CTA is aborting)
            drain_mmas(smem_u32(&sm.acc_done));
        }
    } else if (warp == 3) {
        // this CTA's slice of the array to zero (after pdl_wait above: the
        // kernels before this one are complete)
        if (p.zero != nullptr) {
            const long long ncta = (long long)gridDim.x * gridDim.y * gridDim.z;
            const long long cta = ((long long)blockIdx.z * gridDim.y + blockIdx.y) * gridDim.x + blockIdx.x;
            const long long per = (p.zero_n4 + ncta - 1) / ncta;
            const long long a = cta * per, e = min(p.zero_n4, a + per);
            const float4 z = make_float4(0.f, 0.f, 0.f, 0.f);
            for (long long i = a + lane; i < e; i += 32) p.zero[i] = z;
        }
    } else if (warp >= 4) {
        pdl_trigger();
        const int q = warp & 3, ch = (warp - 4) >> 2;
        const int r = q * 32 + lane;                  // query row of the block; key row at the end
        const uint32_t lane_off = (uint32_t)(q * 32) << 16;
        bool ok = true;
        // dQ of block i (its dK and dQ done; buffer i % 2) into the fp32
        // accumulator: this warp's query rows 32 q .. +31, columns 32 ch .. +31,
        // staged (128-byte swizzled, as the map's swizzle expects) in the rows
        // of dS tile i % 2 this warp itself writes, then one bulk reduce-add
        // issued by lane 0 (rows past k are skipped by the map)
        auto drain_dq = [&](int i) {
            ok = bwait(sm, sm.dq_full[i & 1], (i >> 1) & 1, p.status) && ok;
            tc_fence_after();
            float dq[32];
            tmem_ld32(tDQ + 64 * (i & 1) + lane_off + 32 * ch, dq);
            tc_fence_before();
            mbar_arrive(smem_u32(&sm.dq_empty[i & 1]));
            const bool live = __all_sync(0xffffffffu, ok && !*(volatile int *)&sm.abort);
            if (!live) return;
            uint8_t *xs = sm.ds[i & 1][ch] + q * 4096;
            stage_f32x32(xs, dq, p.scale, lane);   // ends with __syncwarp
            fence_proxy_async();
            __syncwarp();
            const int q0 = (jt + i) * 128 + q * 32;   // first query row of this warp
            if (lane == 0 && q0 < p.k) {
                tma_reduce_add_4d(&p.mDQ, smem_u32(xs), 32 * ch, q0, b, h);
                bulk_commit();
            }
        };
        // this warp's staged dQ rows must have been read before dS overwrites them
        auto staging_read = [&]() {
            if (lane == 0) bulk_wait_read0();
            __syncwarp();
        };
        // lse (log2 units) and D of this thread's query row, one block ahead
        auto row_terms = [&](int i, float &l2, float &dd) {
            const int qi = (jt + i) * 128 + r;
            const bool v = i < nb && qi < p.k;
            l2 = v ? __ldg(p.lse + base + qi) * 1.4426950408889634f : 0.f;
            dd = v ? __ldg(p.Dd + base + qi) : 0.f;
        };
        float l2n, ddn;
        row_terms(0, l2n, ddn);
        for (int i = 0; i < nb; ++i) {
            const int qi = (jt + i) * 128 + r;        // query index
            const bool valid = qi < p.k;
            const float l2 = l2n, dd = ddn;
            row_terms(i + 1, l2n, ddn);
            ok = bwait(sm, sm.sp_full, i & 1, p.status) && ok;
            tc_fence_after();
            // P over this thread's 64 keys (the diagonal block i = 0 is causal)
            float pv[64];
            tmem_ld64(tS + lane_off + 64 * ch, pv);
            tc_fence_before();
            mbar_arrive(smem_u32(&sm.s_free));        // S_{i+1} may overwrite these columns
            if (i == 0 || !valid) {
                // the diagonal block is causal (key offsets c <= lim visible);
                // rows past k see nothing
                const int lim = valid ? r - 64 * ch : -1;
#pragma unroll
                for (int c = 0; c < 64; ++c)
                    pv[c] = c <= lim ? exp2_fast(fmaf(pv[c], p.scale_log2, -l2)) : 0.f;
            } else {
#pragma unroll
                for (int c = 0; c < 64; ++c) pv[c] = exp2_fast(fmaf(pv[c], p.scale_log2, -l2));
            }
            // the P tile holds P_{i-1} until dV_{i-1} has read it
            if (i > 0) {
                ok = bwait(sm, sm.pv_done, (i - 1) & 1, p.status) && ok;
                tc_fence_after();
            }
            put_f16_32(sm.p[ch], r, 0, pv, 1.f);
            put_f16_32(sm.p[ch], r, 32, pv + 32, 1.f);
            fence_proxy_async();
            tc_fence_before();
            mbar_arrive(smem_u32(&sm.p_ready));
            // dQ_{i-2} out: frees its TMEM buffer, and its completion also
            // frees the dS tile this block writes
            if (i >= 2) drain_dq(i - 2);
            // dS = P o (dP - D)
            ok = bwait(sm, sm.dp_full, i & 1, p.status) && ok;
            tc_fence_after();
            {
                float dp[64];
                tmem_ld64(tDP + lane_off + 64 * ch, dp);
#pragma unroll
                for (int c = 0; c < 64; ++c) pv[c] *= dp[c] - dd;
            }
            staging_read();
            put_f16_32(sm.ds[i & 1][ch], r, 0, pv, 1.f);
            put_f16_32(sm.ds[i & 1][ch], r, 32, pv + 32, 1.f);
            fence_proxy_async();
            tc_fence_before();
            mbar_arrive(smem_u32(&sm.ds_ready));       // also: dP_{i+1} may overwrite dP_i
        }
        if (nb >= 2) drain_dq(nb - 2);
        drain_dq(nb - 1);
        if (lane == 0) bulk_wait0();   // the reductions are complete before the CTA's smem goes
        __syncwarp();
        // dK / sqrt(h') and dV of the tile's keys (row r = key j0 + r); an fp16
        // dS out of range has made them non-finite, which flags it
        const bool done = bwait(sm, sm.acc_done, 0, p.status);
        tc_fence_after();
        const int kj = j0 + r;
        const bool live = __all_sync(0xffffffffu, ok && done && !*(volatile int *)&sm.abort) && nb > 0;
        const uint32_t src[2] = {tDK, tDV};
        const float fac[2] = {p.scale, 1.f};
        const int tpos = (p.rope && kj < p.k) ? p.gidx[base + kj] % p.T : 0;
        float vmax = 0.f;   // an out-of-range dS made these non-finite
#pragma unroll
        for (int t = 0; t < 2; ++t) {
            float v[32];
            tmem_ld32(src[t] + lane_off + 32 * ch, v);
            if (!live) continue;
#pragma unroll
            for (int c = 0; c < 32; ++c) v[c] *= fac[t];
            if (t == 0 && p.rope && ch == 0) {
                // dK columns 0..31 are the turned pairs (2p, 2p+1), p < 16
#pragma unroll
                for (int pp = 0; pp < 16; ++pp)
                    rope_turn(v[2 * pp], v[2 * pp + 1], p.rope_tab.phi[pp], tpos, -1.f);
            }
            if (kj < p.k) {
                __half *row = reinterpret_cast<__half *>(p.dQKV) + (base + kj) * 256 + 64 * (t + 1) + 32 * ch;
#pragma unroll
                for (int u = 0; u < 4; ++u) {
                    uint32_t w[4];
#pragma unroll
                    for (int e = 0; e < 4; ++e) {
                        const float a = v[8 * u + 2 * e], c2 = v[8 * u + 2 * e + 1];
                        vmax = fmaxf(vmax, fmaxf(fabsf(a), fabsf(c2)));
                        w[e] = pack_f16x2(a, c2);
                    }
                    reinterpret_cast<uint4 *>(row)[u] = make_uint4(w[0], w[1], w[2], w[3]);
                }
            }
        }
        if (live && kj < p.k && !(vmax < kF16Overflow)) atomicOr(p.status, kStatusRange);
    }
    tc_fence_before();
    __syncthreads();
    span_end(p.span);
    if (warp == 2) {
        tc_fence_after();
        tmem_dealloc(tmem, 512);
    }
}

// dQ from its fp32 accumulator into columns 0..63 of the dQ|dK|dV|dlogit rows,
// eight columns per thread (two 16-byte loads): as a bf16 pair ([hi 256 | lo
// 256] rows), or (f16) as fp16 rows of 256 (one 16-byte store), turned back by
// RoPE first when asked (gidx, rope).
__global__ void dq_finish_kernel(const float *__restrict__ dQacc, bf16 *__restrict__ dQKV, size_t rows,
                                 int f16, const int32_t *__restrict__ gidx, int rope, int T,
                                 RopeTable tab, uint32_t *status, unsigned long long *span) {
    pdl_trigger();  // the next kernel (zeroing dX) may run beside this one
    pdl_wait();
    span_begin(span);
    const size_t idx = (size_t)blockIdx.x * blockDim.x + threadIdx.x;   // (row, 8-column group)
    if (idx >= rows * 8) return;
    const size_t row = idx >> 3;
    const int c = (int)(idx & 7) * 8;
    const float4 a = *reinterpret_cast<const float4 *>(dQacc + row * 64 + c);
    const float4 b = *reinterpret_cast<const float4 *>(dQacc + row * 64 + c + 4);
    float v[8] = {a.x, a.y, a.z, a.w, b.x, b.y, b.z, b.w};
    if (!f16) {
        uint32_t hi[4], lo[4];
#pragma unroll
        for (int e = 0; e < 4; ++e) split_pair2(v[2 * e], v[2 * e + 1], hi[e], lo[e]);
        *reinterpret_cast<uint4 *>(dQKV + row * 512 + c) = make_uint4(hi[0], hi[1], hi[2], hi[3]);
        *reinterpret_cast<uint4 *>(dQKV + row * 512 + 256 + c) = make_uint4(lo[0], lo[1], lo[2], lo[3]);
        return;
    }
    if (rope && c < 32) {
        const int t = gidx[row] % T;
#pragma unroll
        for (int e = 0; e < 4; ++e) rope_turn(v[2 * e], v[2 * e + 1], tab.phi[(c >> 1) + e], t, -1.f);
    }
    uint32_t w[4];
    float mx = 0.f;
#pragma unroll
    for (int e = 0; e < 4; ++e) {
        mx = fmaxf(mx, fmaxf(fabsf(v[2 * e]), fabsf(v[2 * e + 1])));
        w[e] = pack_f16x2(v[2 * e], v[2 * e + 1]);
    }
    *reinterpret_cast<uint4 *>(reinterpret_cast<__half *>(dQKV) + row * 256 + c) = make_uint4(w[0], w[1], w[2], w[3]);
    if (!(mx < kF16Overflow)) atomicOr(status, kStatusRange);
    span_end(span);   // (thread 0 of each block, after its own row group)
}

// ------------------------------------------------- k <= 128: one CTA per tile
// When a head keeps at most 128 tokens the whole k x k problem of one (b, h)
// unit fits one CTA: a single 128-key block, no online rescaling (forward) and
// one fused pass for dQ, dK and dV (backward).  U = floor(128 / k) consecutive
// sequences of the same head share the tile (their rows are adjacent in the
// [H, B*k] layout); the mask is then block-diagonal and causal within each
// block.  P (then dS) lives in one 128 x 128 bf16-pair tile: K-major (keys
// contiguous) for P V and dS K, and read through an MN-major descriptor as
// P^T / dS^T for dV and dK.

constexpr int kSmallK = 128;
constexpr int kPBig = kTileHalf;   // one 64-key block of a 128-row tile, one half: 16 KB

struct SmallFwdSmem {
    uint8_t q[2][kPBig];
    uint8_t k[2][kPBig];
    uint8_t v[2][kPBig];
    uint8_t p[2][2][kPBig];           // [half][key block]
    float part_max[2][128], part_sum[2][128];   // per key half: row max, row sum
    uint64_t in_full, s_full, p_ready, o_full;
    uint32_t tmem;
    int abort;
};
constexpr int kSmallFwdSmem = (int)sizeof(SmallFwdSmem) + 1024;

struct SmallBwdSmem {
    uint8_t q[2][kPBig];
    uint8_t k[2][kPBig];
    uint8_t v[2][kPBig];
    uint8_t da[2][kPBig];
    uint8_t p[2][2][kPBig];           // P, then dS
    uint64_t in_full, sp_full, p_ready, pv_done, ds_ready, acc_done;
    uint32_t tmem;
    int abort;
};
constexpr int kSmallBwdSmem = (int)sizeof(SmallBwdSmem) + 1024;

// Threads of the k <= 128 kernels: warps 0-3 load, issue MMAs and own TMEM;
// warps 4-11 run the softmax passes and the epilogue, two per TMEM lane
// quadrant: warp w serves tile rows 32 (w % 4) .. +31 and key (or output)
// column half ch = (w - 4) / 4.
constexpr int kSmallThreads = 384;
constexpr int kSoftmaxThreads = 256;

__global__ void __launch_bounds__(kSmallThreads, 1) attn_fwd_small_kernel(const __grid_constant__ AttnParams p) {
    extern __shared__ uint8_t smem_raw[];
    SmallFwdSmem &sm = *reinterpret_cast<SmallFwdSmem *>(
        (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int b0 = blockIdx.y * p.U, h = blockIdx.z;
    if (threadIdx.x == 0) {
        mbar_init(smem_u32(&sm.in_full), 1);
        mbar_init(smem_u32(&sm.s_full), 1);
        mbar_init(smem_u32(&sm.p_ready), kSoftmaxThreads);
        mbar_init(smem_u32(&sm.o_full), 1);
        sm.abort = 0;
        fence_barrier_init();
    }
    if (warp == 2) {
        tmem_alloc(smem_u32(&sm.tmem), 256);
        tmem_relinquish();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    pdl_wait();  // Q, K, V, dA, lse written by the previous kernels
    span_begin(p.span);
    const uint32_t tmem = sm.tmem, tS = tmem, tO = tmem + 128;

    if (warp == 0) {
        if (lane == 0) {
            const uint32_t fb = smem_u32(&sm.in_full);
            mbar_expect_tx(fb, 6 * kPBig);
            for (int hf = 0; hf < 2; ++hf) {
                tma_load_3d(smem_u32(sm.q[hf]), &p.mQ, fb, 64 * hf, b0 * p.k, h);
                tma_load_3d(smem_u32(sm.k[hf]), &p.mK, fb, 64 * hf, b0 * p.k, h);
                tma_load_3d(smem_u32(sm.v[hf]), &p.mV, fb, 64 * hf, b0 * p.k, h);
            }
            drain_phase(fb, 0);
        }
    } else if (warp == 1) {
        if (lane == 0) {
            constexpr uint32_t idS = idesc_bf16(128, 128, false, false);
            constexpr uint32_t idO = idesc_bf16(128, 64, false, true);
            bool ok = mbar_wait(smem_u32(&sm.in_full), 0);
            if (ok) {
                tc_fence_after();
                // S = Q K^T: K (keys x p) is the K-major B operand, N = 128 keys
                const uint32_t qa[3] = {smem_u32(sm.q[0]), smem_u32(sm.q[0]), smem_u32(sm.q[1])};
                const uint32_t kb[3] = {smem_u32(sm.k[0]), smem_u32(sm.k[1]), smem_u32(sm.k[0])};
#pragma unroll
                for (int t = 0; t < 3; ++t)
#pragma unroll
                    for (int kk = 0; kk < 4; ++kk)
                        mma_bf16(tS, smem_desc_sw128(qa[t] + kk * 32, 16, 1024),
                                 smem_desc_sw128(kb[t] + kk * 32, 16, 1024), idS,
                                 (t > 0 || kk > 0) ? 1u : 0u);
                mma_commit(smem_u32(&sm.s_full));
                ok = mbar_wait(smem_u32(&sm.p_ready), 0) && !*(volatile int *)&sm.abort;
                if (ok) {
                    tc_fence_after();
                    mma_k128(tO, sm.p, sm.v, false, idO);
                }
            }
            if (!ok) {
                flag_timeout_b(sm, p.status);
                mma_commit(smem_u32(&sm.s_full));   // release the softmax warps
            }
            drain_mmas(smem_u32(&sm.o_full));   // o_full's only phase covers every MMA
        }
    } else if (warp >= 4) {
        pdl_trigger();
        const int q = warp & 3, ch = (warp - 4) >> 2;
        const int r = q * 32 + lane;   // query row i of the tile
        const int cb = 64 * ch;        // this thread's 64 keys
        const TileRow tr = tile_row(r, p.k, p.U, b0, p.B);
        const int lo = tr.valid ? tr.lo : r + 1;   // invalid rows see no keys
        const uint32_t lane_off = (uint32_t)(q * 32) << 16;
        bool ok = mbar_wait(smem_u32(&sm.s_full), 0);
        tc_fence_after();
        // pass 1: row max over both halves
        float m = -INFINITY;
#pragma unroll 1
        for (int c0 = cb; c0 < cb + 64; c0 += 32) {
            float t32[32];
            tmem_ld32(tS + lane_off + c0, t32);
#pragma unroll
            for (int c = 0; c < 32; ++c)
                if (c0 + c <= r && c0 + c >= lo) m = fmaxf(m, t32[c] * p.scale_log2);
        }
        sm.part_max[ch][r] = m;
        named_barrier(1, kSoftmaxThreads);
        m = fmaxf(sm.part_max[0][r], sm.part_max[1][r]);
        // pass 2: probabilities into shared memory, partial row sums
        float l = 0.f;
#pragma unroll 1
        for (int c0 = cb; c0 < cb + 64; c0 += 32) {
            float t32[32];
            tmem_ld32(tS + lane_off + c0, t32);
#pragma unroll
            for (int c = 0; c < 32; ++c) {
                t32[c] = (c0 + c <= r && c0 + c >= lo) ? exp2_fast(t32[c] * p.scale_log2 - m) : 0.f;
                l += t32[c];
            }
            write_pair32(sm.p, r, c0, t32);
        }
        sm.part_sum[ch][r] = l;
        fence_proxy_async();
        tc_fence_before();
        mbar_arrive(smem_u32(&sm.p_ready));
        ok = mbar_wait(smem_u32(&sm.o_full), 0) && ok;
        tc_fence_after();
        named_barrier(1, kSoftmaxThreads);   // partial sums visible
        l = sm.part_sum[0][r] + sm.part_sum[1][r];
        float o[32];
        tmem_ld32(tO + lane_off + 32 * ch, o);   // output columns 32 ch .. 32 ch + 31
        if (!ok) flag_timeout_b(sm, p.status);
        const bool live = __all_sync(0xffffffffu, ok && !*(volatile int *)&sm.abort);
        const unsigned vmask = __ballot_sync(0xffffffffu, tr.valid);
        const size_t row0 = (size_t)h * p.Mtok + (size_t)b0 * p.k + q * 32;   // global row of lane 0
        if (live) {
            // Q tile is free once S is done: 4 KB of staging per softmax warp
            uint8_t *xb = sm.q[0] + (warp - 4) * 4096;
            const float inv = tr.valid ? 1.f / l : 0.f;
            const float rr = tr.valid ? p.rsel[row0 + lane] : 0.f;
            stage_pair32(xb, o, inv * rr, lane);
            store_rows128(xb, lane, [&](int rl, int c) -> uint4 * {
                if (!((vmask >> rl) & 1u)) return nullptr;
                bf16 *base = p.AR + (row0 + rl) * 128 + 32 * ch;
                return c < 4 ? reinterpret_cast<uint4 *>(base) + c
                             : reinterpret_cast<uint4 *>(base + 64) + (c - 4);
            });
            // lse in natural-log units of the scaled scores
            if (ch == 0 && tr.valid) p.lse[row0 + lane] = (m + log2f(l)) * 0.69314718055994531f;
        }
    }
    tc_fence_before();
    __syncthreads();
    span_end(p.span);
    if (warp == 2) {
        tc_fence_after();
        tmem_dealloc(tmem, 256);
    }
}

__global__ void __launch_bounds__(kSmallThreads, 1) attn_bwd_small_kernel(const __grid_constant__ BwdParams p) {
    extern __shared__ uint8_t smem_raw[];
    SmallBwdSmem &sm = *reinterpret_cast<SmallBwdSmem *>(
        (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int b0 = blockIdx.y * p.U, h = blockIdx.z;
    if (threadIdx.x == 0) {
        mbar_init(smem_u32(&sm.in_full), 1);
        mbar_init(smem_u32(&sm.sp_full), 1);
        mbar_init(smem_u32(&sm.p_ready), kSoftmaxThreads);
        mbar_init(smem_u32(&sm.pv_done), 1);
        mbar_init(smem_u32(&sm.ds_ready), kSoftmaxThreads);
        mbar_init(smem_u32(&sm.acc_done), 1);
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
    pdl_wait();  // Q, K, V, dA, lse written by the previous kernels
    span_begin(p.span);
    const uint32_t tmem = sm.tmem;
    const uint32_t tS = tmem, tDP = tmem + 128, tDV = tmem + 256, tDK = tmem + 320, tDQ = tmem + 384;

    if (warp == 0) {
        if (lane == 0) {
            const uint32_t fb = smem_u32(&sm.in_full);
            mbar_expect_tx(fb, 8 * kPBig);
            for (int hf = 0; hf < 2; ++hf) {
                tma_load_3d(smem_u32(sm.q[hf]), &p.mA0, fb, 64 * hf, b0 * p.k, h);
                tma_load_3d(smem_u32(sm.k[hf]), &p.mA1, fb, 64 * hf, b0 * p.k, h);
                tma_load_3d(smem_u32(sm.v[hf]), &p.mB0, fb, 64 * hf, b0 * p.k, h);
                tma_load_3d(smem_u32(sm.da[hf]), &p.mB1, fb, 64 * hf, b0 * p.k, h);
            }
            drain_phase(fb, 0);
        }
    } else if (warp == 1) {
        if (lane == 0) {
            constexpr uint32_t idKK = idesc_bf16(128, 128, false, false);  // S, dP
            constexpr uint32_t idMN = idesc_bf16(128, 64, true, true);     // dV, dK
            constexpr uint32_t idKM = idesc_bf16(128, 64, false, true);    // dQ
            bool ok = mbar_wait(smem_u32(&sm.in_full), 0);
            if (ok) {
                tc_fence_after();
                const uint32_t q0 = smem_u32(sm.q[0]), q1 = smem_u32(sm.q[1]);
                const uint32_t k0 = smem_u32(sm.k[0]), k1 = smem_u32(sm.k[1]);
                const uint32_t v0 = smem_u32(sm.v[0]), v1 = smem_u32(sm.v[1]);
                const uint32_t a0 = smem_u32(sm.da[0]), a1 = smem_u32(sm.da[1]);
                mma_pair3(tS, q0, q1, k0, k1, false, false, idKK, false);   // S  = Q K^T
                mma_pair3(tDP, a0, a1, v0, v1, false, false, idKK, false);  // dP = dA V^T
                mma_commit(smem_u32(&sm.sp_full));
                ok = mbar_wait(smem_u32(&sm.p_ready), 0) && !*(volatile int *)&sm.abort;
                if (ok) {
                    tc_fence_after();
                    mma_k128(tDV, sm.p, sm.da, true, idMN);   // dV = P^T dA
                    mma_commit(smem_u32(&sm.pv_done));
                    ok = mbar_wait(smem_u32(&sm.ds_ready), 0) && !*(volatile int *)&sm.abort;
                }
                if (ok) {
                    tc_fence_after();
                    mma_k128(tDK, sm.p, sm.q, true, idMN);    // dK = dS^T Q
                    mma_k128(tDQ, sm.p, sm.k, false, idKM);   // dQ = dS K
                }
            }
            if (!ok) {
                flag_timeout_b(sm, p.status);
                mma_commit(smem_u32(&sm.sp_full));
                mma_commit(smem_u32(&sm.pv_done));
            }
            drain_mmas(smem_u32(&sm.acc_done));   // acc_done's only phase covers every MMA
        }
    } else if (warp >= 4) {
        pdl_trigger();
        const int q = warp & 3, ch = (warp - 4) >> 2;
        const int r = q * 32 + lane;   // query row i for S/dP/dQ; key row j for dK/dV
        const int cb = 64 * ch;        // this thread's 64 keys
        const uint32_t lane_off = (uint32_t)(q * 32) << 16;
        const size_t base = (size_t)h * p.Mtok + (size_t)b0 * p.k;
        const TileRow tr = tile_row(r, p.k, p.U, b0, p.B);
        const bool valid = tr.valid;
        const int lo = tr.lo;
        const float l2 = valid ? p.lse[base + r] * 1.4426950408889634f : 0.f;
        const float dd = valid ? p.Dd[base + r] : 0.f;
        bool ok = mbar_wait(smem_u32(&sm.sp_full), 0);
        tc_fence_after();
        // P
#pragma unroll 1
        for (int c0 = cb; c0 < cb + 64; c0 += 32) {
            float t32[32];
            tmem_ld32(tS + lane_off + c0, t32);
#pragma unroll
            for (int c = 0; c < 32; ++c)
                t32[c] = (valid && c0 + c <= r && c0 + c >= lo) ? exp2_fast(t32[c] * p.scale_log2 - l2) : 0.f;
            write_pair32(sm.p, r, c0, t32);
        }
        fence_proxy_async();
        tc_fence_before();
        mbar_arrive(smem_u32(&sm.p_ready));
        ok = mbar_wait(smem_u32(&sm.pv_done), 0) && ok;   // P read by dV: overwrite with dS
        tc_fence_after();
#pragma unroll 1
        for (int c0 = cb; c0 < cb + 64; c0 += 32) {
            float t32[32], d32[32];
            tmem_ld32(tS + lane_off + c0, t32);
            tmem_ld32(tDP + lane_off + c0, d32);
#pragma unroll
            for (int c = 0; c < 32; ++c) {
                const float pr = (valid && c0 + c <= r && c0 + c >= lo) ? exp2_fast(t32[c] * p.scale_log2 - l2) : 0.f;
                t32[c] = pr * (d32[c] - dd);
            }
            write_pair32(sm.p, r, c0, t32);
        }
        fence_proxy_async();
        tc_fence_before();
        mbar_arrive(smem_u32(&sm.ds_ready));
        ok = mbar_wait(smem_u32(&sm.acc_done), 0) && ok;
        tc_fence_after();
        if (!ok) flag_timeout_b(sm, p.status);
        const bool live = __all_sync(0xffffffffu, ok && !*(volatile int *)&sm.abort);
        // dQ, dK, dV columns 32 ch .. +31 into the Q, K, V tiles (free once
        // every MMA is done), then out by TMA stores into the dQKV rows: as
        // bf16 pairs (hi blocks at columns 0, 64, 128, lo blocks 256 further)
        // or as single fp16 blocks at columns 0, 64, 128
        uint8_t(*tiles[3])[kPBig] = {sm.q, sm.k, sm.v};
        const uint32_t src[3] = {tDQ, tDK, tDV};
        const float fac[3] = {p.scale, p.scale, 1.f};
        // original position of this row's token (RoPE is turned back on the
        // first 32 columns of dQ and dK, which only ch == 0 holds)
        const int tpos = (p.out16 && p.rope && valid && ch == 0) ? p.gidx[base + r] % p.T : 0;
        float omax = 0.f;
#pragma unroll 1
        for (int t = 0; t < 3; ++t) {
            float v[32];
            tmem_ld32(src[t] + lane_off + 32 * ch, v);
            if (!p.out16) {
                put_pair32(tiles[t][0], tiles[t][1], r, 32 * ch, v, fac[t]);
                continue;
            }
            if (p.rope && t < 2 && ch == 0) {
#pragma unroll
                for (int pp = 0; pp < 16; ++pp)
                    rope_turn(v[2 * pp], v[2 * pp + 1], p.rope_tab.phi[pp], tpos, -1.f);
            }
            omax = fmaxf(omax, put_f16_32(tiles[t][0], r, 32 * ch, v, fac[t]));
        }
        if (p.out16 && live && valid && !(omax < kF16Overflow)) atomicOr(p.status, kStatusRange);
        fence_proxy_async();
        named_barrier(1, kSoftmaxThreads);
        if (threadIdx.x == 128 && live) {
            for (int t = 0; t < 3; ++t)
                for (int hf = 0; hf < (p.out16 ? 1 : 2); ++hf)
                    tma_store_3d(&p.mOut, smem_u32(tiles[t][hf]), 64 * t + 256 * hf, b0 * p.k, h);
            bulk_commit();
            bulk_wait0();
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

bool map_rows(CUtensorMap *m, const void *base, int H, int Mtok) {
    // [H, B*k, 128] bf16 pair array, box {64, 128, 1}: 128 consecutive rows of one head
    const uint64_t dims[3] = {128, (uint64_t)Mtok, (uint64_t)H};
    const uint64_t strides[2] = {256, (uint64_t)Mtok * 256};
    const uint32_t box[3] = {64, 128, 1};
    return tmap_bf16(m, base, 3, dims, strides, box);
}

// [H, B, k, 64] fp16 array (k > 128 path), box {64, rows, 1, 1}: rows past k
// of one sequence read as zeros.  (The map's element type only sets the
// element size; the tiles are copied bit for bit.)
bool map_units(CUtensorMap *m, const void *base, int H, int B, int k, uint32_t rows) {
    const uint64_t dims[4] = {64, (uint64_t)k, (uint64_t)B, (uint64_t)H};
    const uint64_t strides[3] = {128, (uint64_t)k * 128, (uint64_t)B * k * 128};
    const uint32_t box[4] = {64, rows, 1, 1};
    return tmap_bf16(m, base, 4, dims, strides, box);
}

}  // namespace

cudaError_t tc_attn_fwd(const Dims &dm, const Saved &sv, cudaStream_t s) {
    AttnParams p;
    memset(&p, 0, sizeof(p));
    const bool small = dm.k <= kSmallK;
    const int Mtok = dm.B * dm.k;
    bool ok = small ? (map_rows(&p.mQ, sv.Q, dm.H, Mtok) && map_rows(&p.mK, sv.K, dm.H, Mtok) &&
                       map_rows(&p.mV, sv.V, dm.H, Mtok))
                    : (map_units(&p.mQ, sv.Q, dm.H, dm.B, dm.k, kQ) &&
                       map_units(&p.mK, sv.K, dm.H, dm.B, dm.k, kLKeys) &&
                       map_units(&p.mV, sv.V, dm.H, dm.B, dm.k, kLKeys));
    if (!ok) return cudaErrorInvalidValue;
    p.U = small ? kSmallK / dm.k : 1;
    p.k = dm.k;
    p.B = dm.B;
    p.Mtok = dm.B * dm.k;
    p.scale_log2 = 1.4426950408889634f / sqrtf(64.f);
    p.rsel = sv.rsel;
    p.AR = static_cast<bf16 *>(sv.AR);
    p.AR16 = small ? nullptr : static_cast<__half *>(sv.AR16);
    p.lse = sv.lse;
    p.status = sv.status;
    p.span = active_span();
    cudaError_t attr = allow_smem((const void *)attn_fwd_tc_kernel, kFwdLargeSmem);
    if (attr == cudaSuccess) attr = allow_smem((const void *)attn_fwd_small_kernel, kSmallFwdSmem);
    if (attr != cudaSuccess) return attr;
    if (small) {
        cudaError_t e = launch_pdl(attn_fwd_small_kernel, dim3(1, (dm.B + p.U - 1) / p.U, dm.H),
                                   dim3(kSmallThreads), kSmallFwdSmem, s, p);
        note_launches(1);
        return e;
    }
    dim3 grid(dm.B, dm.H, (dm.k + kQ - 1) / kQ);   // query tiles slowest (see the kernel)
    cudaError_t e = launch_pdl(attn_fwd_tc_kernel, grid, dim3(kLT), kFwdLargeSmem, s, p);
    note_launches(1);
    return e;
}

cudaError_t tc_attn_bwd(const Dims &dm, const Saved &sv, cudaStream_t s, float *zero_out) {
    BwdParams kv, dq;
    memset(&kv, 0, sizeof(kv));
    memset(&dq, 0, sizeof(dq));
    if (dm.k <= kSmallK) {
        BwdParams sp;
        memset(&sp, 0, sizeof(sp));
        const int Mtok = dm.B * dm.k;
        sp.U = kSmallK / dm.k;
        // dQ|dK|dV|dlogit rows: fp16 [H, B*k, 256], or bf16 pairs [H, B*k, 512]
        sp.out16 = dqkv_f16(dm) ? 1 : 0;
        const uint64_t ocols = sp.out16 ? 256 : 512;
        const uint64_t odims[3] = {ocols, (uint64_t)Mtok, (uint64_t)dm.H};
        const uint64_t ostrides[2] = {ocols * 2, (uint64_t)Mtok * ocols * 2};
        const uint32_t obox[3] = {64, (uint32_t)(sp.U * dm.k), 1};
        const bool ok = map_rows(&sp.mA0, sv.Q, dm.H, Mtok) && map_rows(&sp.mA1, sv.K, dm.H, Mtok) &&
                        map_rows(&sp.mB0, sv.V, dm.H, Mtok) && map_rows(&sp.mB1, sv.dA, dm.H, Mtok) &&
                        tmap_bf16(&sp.mOut, sv.dQKV, 3, odims, ostrides, obox);
        if (!ok) return cudaErrorInvalidValue;
        sp.B = dm.B;
        sp.k = dm.k;
        sp.Mtok = dm.B * dm.k;
        sp.scale = 1.f / sqrtf(64.f);
        sp.scale_log2 = 1.4426950408889634f / sqrtf(64.f);
        sp.lse = sv.lse;
        sp.Dd = sv.Dd;
        sp.dQKV = static_cast<bf16 *>(sv.dQKV);
        sp.status = sv.status;
        sp.span = active_span();
        sp.gidx = sv.gidx;
        sp.T = dm.T;
        sp.rope = dm.rope ? 1 : 0;
        if (dm.rope) sp.rope_tab = make_rope_table(dm.hp, dm.T);
        const cudaError_t attr_small = allow_smem((const void *)attn_bwd_small_kernel, kSmallBwdSmem);
        if (attr_small != cudaSuccess) return attr_small;
        cudaError_t e = launch_pdl(attn_bwd_small_kernel, dim3(1, (dm.B + sp.U - 1) / sp.U, dm.H),
                                   dim3(kSmallThreads), kSmallBwdSmem, s, sp);
        note_launches(1);
        return e;
    }
    // k > 128: one CTA per 128-key tile; dQ accumulates in fp32 (the
    // workspace's G buffer, unused on this path) and is split into pairs after
    BwdParams bp;
    memset(&bp, 0, sizeof(bp));
    bool ok = map_units(&bp.mA0, sv.K, dm.H, dm.B, dm.k, 128) &&
              map_units(&bp.mA1, sv.V, dm.H, dm.B, dm.k, 128) &&
              map_units(&bp.mB0, sv.Q, dm.H, dm.B, dm.k, 128) &&
              map_units(&bp.mB1, sv.dA, dm.H, dm.B, dm.k, 128);
    if (!ok) return cudaErrorInvalidValue;
    bp.k = dm.k;
    bp.Mtok = dm.B * dm.k;
    bp.scale = 1.f / sqrtf(64.f);
    bp.scale_log2 = 1.4426950408889634f / sqrtf(64.f);
    bp.lse = sv.lse;
    bp.Dd = sv.Dd;
    bp.dQKV = static_cast<bf16 *>(sv.dQKV);
    bp.dQacc = sv.G;
    bp.status = sv.status;
    bp.span = active_span();
    bp.gidx = sv.gidx;
    bp.T = dm.T;
    bp.rope = dm.rope ? 1 : 0;
    if (dm.rope) bp.rope_tab = make_rope_table(dm.hp, dm.T);
    if (zero_out != nullptr) {
        bp.zero = reinterpret_cast<float4 *>(zero_out);
        bp.zero_n4 = (long long)dm.B * dm.T * dm.d / 4;
    }
    {
        // dQ accumulator [H, B, k, 64] fp32 (the workspace's G buffer)
        const uint64_t dims[4] = {64, (uint64_t)dm.k, (uint64_t)dm.B, (uint64_t)dm.H};
        const uint64_t strides[3] = {256, (uint64_t)dm.k * 256, (uint64_t)dm.B * dm.k * 256};
        const uint32_t box[4] = {32, 32, 1, 1};
        if (!tmap_f32(&bp.mDQ, sv.G, 4, dims, strides, box)) return cudaErrorInvalidValue;
    }
    const size_t rows = (size_t)dm.H * dm.B * dm.k;
    const cudaError_t attr = allow_smem((const void *)attn_bwd_tc_kernel, kBwdLargeSmem);
    if (attr != cudaSuccess) return attr;
    // (the dQ accumulator sv.G has been zeroed by the G kernel before this)
    dim3 grid(dm.B, dm.H, (dm.k + 127) / 128);   // key tiles slowest (see the kernel)
    cudaError_t e = launch_pdl(attn_bwd_tc_kernel, grid, dim3(kBT), kBwdLargeSmem, s, bp);
    const size_t n = rows * 8;
    if (e == cudaSuccess)
        e = launch_pdl(dq_finish_kernel, dim3((unsigned)((n + 255) / 256)), dim3(256), 0, s,
                       (const float *)sv.G, static_cast<bf16 *>(sv.dQKV), rows, 1,
                       (const int32_t *)sv.gidx, bp.rope, dm.T, bp.rope_tab, sv.status, bp.span);
    note_launches(2);
    return e;
}

}  // namespace mosa
