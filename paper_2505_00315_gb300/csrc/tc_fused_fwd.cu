// Fused forward of the selected-token path for k <= 128 (Sec. 2.2, Eq.
// mosa_mha: X^s = X[I], Q/K/V = X^s W, causal attention among the k selected
// tokens, X^o = diag(r^topk) A W_o scattered back into the T positions).
//
// One CTA per 128-row tile of one head: U = floor(128 / k) consecutive
// sequences b0 .. b0+U-1 (their rows are adjacent in the [H, B*k] layout), all
// on the tensor cores with fp32 accumulators in TMEM:
//   phase 1  [Q|K|V] = X[g(m), :] [W_q|W_k|W_v][h]   K = d in 64-wide blocks, a
//            5-stage ring (three slots of its own, two in the Q/K/V tiles, idle
//            until phase 2): W blocks by TMA, the selected rows of X by 16-byte
//            cp.async gathers, confirmed three blocks after issue
//   phase 2  the accumulator is read back (Q and K turned by RoPE at the rows'
//            original positions when asked, Sec. 2.2) and split into bf16 hi/lo pairs, kept
//            in shared memory as the attention operands; warp 3 copies them to
//            global memory (the backward reads them) by TMA stores while the
//            softmax runs
//   phase 3  S = Q K^T, block-diagonal causal softmax (two threads per row),
//            O = P V; lse goes to global memory; AR = r A / l (a pair) stays in
//            shared memory and warp 3 stores it by TMA (the backward needs A
//            only through AR)
//   phase 4  Y[g(m), n] += (AR W_o[h])(m, n) for n in 256-wide chunks, W_o
//            chunks double-buffered by TMA, accumulators double-buffered in
//            TMEM so one chunk's scatter-add overlaps the next chunk's MMAs.
// Products with one pair operand are two MMAs, with two pair operands three
// (hi hi + hi lo + lo hi), as in the separate kernels.
//
// Warps: 0 TMA producer, 1 MMA issuer, 2 TMEM owner, 3 TMA stores; 4-11 gather,
// softmax and epilogues, two per TMEM lane quadrant (warp w serves tile rows
// 32 (w % 4) .. +31 and column half (w - 4) / 4).  Every wait is bounded.
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
constexpr int kWorkers = 256;            // warps 4-11
constexpr int kStages = 5;                // ring slots in phase 1
constexpr int kOwnStages = 3;             // slots of the ring array; the others lie in the Q/K/V tiles
constexpr int kLag = kStages - 2;         // gather blocks in flight before one is confirmed
constexpr int kHalf = kTileHalf;         // one hi or lo half of a 128 x 64 tile: 16 KB
constexpr int kStageBytes = kHalf + 3 * 8192;   // gathered X block + W_q|W_k|W_v blocks
constexpr int kChunk = 256;              // output columns per phase-4 chunk

struct FusedSmem {
    // phase 1: the ring; phase 3: P pair tile [half][key block] in its first
    // 64 KB and epilogue staging at +64 KB; phase 4: staging at +64 KB
    uint8_t ring[kOwnStages][kStageBytes];
    uint8_t q[2][kHalf];     // Q pair; phase 4: AR pair (A operand of the output product)
    uint8_t k[2][kHalf];     // K pair; phase 4: W_o chunk buffer 0
    uint8_t v[2][kHalf];     // V pair; phase 4: W_o chunk buffer 1
    float part_max[2][128], part_sum[2][128];
    int rows[128];           // b*T + I of each tile row, -1 for rows outside the tile's sequences
    uint64_t full[kStages], empty[kStages];
    uint64_t qkv_done, qkv_staged, qkv_read, s_full, p_ready, o_full, ar_ready;
    uint64_t wo_full[2], wo_empty[2], out_full[2], out_empty[2];
    uint64_t drained;   // the MMA issuer's final drain
    uint32_t tmem;
    int abort;
};
constexpr int kSmem = (int)sizeof(FusedSmem) + 1024;
static_assert(kSmem <= 227 * 1024, "shared memory");
static_assert((kStages - kOwnStages) * kStageBytes <= 6 * kHalf, "ring slots in the Q/K/V tiles");

struct FusedParams {
    CUtensorMap mW[3];     // W_q, W_k, W_v: [H, d, 64], box {64, 64, 1}
    CUtensorMap mWo;       // W_o: [H, 64, d], box {64, 64, 1}
    CUtensorMap mOut[4];   // Q, K, V, AR pairs: [H, B*k, 128], box {64, U k, 1} (stores)
    const bf16 *X;         // [B*T, d]
    const int32_t *gidx;   // [H, B*k]
    const float *rsel;     // [H, B*k]
    float *lse;            // [H, B*k]
    float *Y;              // [B*T, d], accumulated into
    int B, T, d, k, U, Mtok;
    float scale_log2;
    int rope_on;           // RoPE on Q and K (Sec. 2.2)
    RopeTable rope;
    uint32_t *status;
    unsigned long long *span;   // measurement: kernel span slot, or null
};

// Bounded wait that gives up at once when the CTA is already aborting.
__device__ __forceinline__ bool wait_or_abort(FusedSmem &sm, uint64_t &bar, uint32_t parity,
                                              uint32_t *status) {
    if (*(volatile int *)&sm.abort) return false;
    if (mbar_wait(smem_u32(&bar), parity)) return true;
    atomicOr(status, kStatusTimeout);
    *(volatile int *)&sm.abort = 1;
    return false;
}

__global__ void __launch_bounds__(kThreads, 1) fused_fwd_kernel(const __grid_constant__ FusedParams p) {
    extern __shared__ uint8_t smem_raw[];
    FusedSmem &sm = *reinterpret_cast<FusedSmem *>(
        (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int b0 = blockIdx.x * p.U, h = blockIdx.y;
    const int nkb = (p.d + 63) / 64;
    const int nch = (p.d + kChunk - 1) / kChunk;
    const size_t row_base = (size_t)h * p.Mtok + (size_t)b0 * p.k;  // head row of tile row 0
    // P pair tile [half][key block] over the start of the ring
    uint8_t(*ptile)[2][kHalf] = reinterpret_cast<uint8_t(*)[2][kHalf]>(&sm.ring[0][0]);
    uint8_t *stage_area = &sm.ring[0][0] + 4 * kHalf;   // 32 KB of epilogue staging
    // phase-1 ring slot s: the ring array, then the Q/K/V tiles (contiguous, idle
    // until the Q|K|V product is done)
    auto slot = [&](int s) -> uint8_t * {
        return s < kOwnStages ? sm.ring[s] : &sm.q[0][0] + (s - kOwnStages) * kStageBytes;
    };

    if (threadIdx.x == 0) {
        for (int s = 0; s < kStages; ++s) {
            mbar_init(smem_u32(&sm.full[s]), 1 + kWorkers);
            mbar_init(smem_u32(&sm.empty[s]), 1);
        }
        mbar_init(smem_u32(&sm.qkv_done), 1);
        mbar_init(smem_u32(&sm.qkv_staged), kWorkers);
        mbar_init(smem_u32(&sm.qkv_read), 1);
        mbar_init(smem_u32(&sm.s_full), 1);
        mbar_init(smem_u32(&sm.p_ready), kWorkers);
        mbar_init(smem_u32(&sm.o_full), 1);
        mbar_init(smem_u32(&sm.ar_ready), kWorkers);
        for (int i = 0; i < 2; ++i) {
            mbar_init(smem_u32(&sm.wo_full[i]), 1);
            mbar_init(smem_u32(&sm.wo_empty[i]), 1);
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
    pdl_wait();  // gidx and r_sel come from the selection kernel
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
            int issued = 0, nc = 0;   // ring stages and W_o chunks loaded
            for (int kb = 0; kb < nkb; ++kb) {
                const int s = kb % kStages;
                if (!wait_or_abort(sm, sm.empty[s], ((kb / kStages) & 1) ^ 1, p.status)) break;
                const uint32_t fb = smem_u32(&sm.full[s]);
                mbar_expect_tx(fb, 3 * 8192);
                for (int j = 0; j < 3; ++j)
                    tma_load_3d(smem_u32(slot(s) + kHalf + j * 8192), &p.mW[j], fb, 0, kb * 64, h);
                issued = kb + 1;
            }
            // phase 4: W_o chunks into the K / V tiles once P V is done and
            // their TMA stores have read them
            if (wait_or_abort(sm, sm.o_full, 0, p.status) &&
                wait_or_abort(sm, sm.qkv_read, 0, p.status)) {
                for (int c = 0; c < nch; ++c) {
                    const int buf = c & 1;
                    if (c >= 2 && !wait_or_abort(sm, sm.wo_empty[buf], ((c >> 1) - 1) & 1, p.status))
                        break;
                    const uint32_t fb = smem_u32(&sm.wo_full[buf]);
                    uint8_t *dst = buf ? &sm.v[0][0] : &sm.k[0][0];
                    mbar_expect_tx(fb, 4 * 8192);
                    for (int j = 0; j < 4; ++j)
                        tma_load_3d(smem_u32(dst + j * 8192), &p.mWo, fb, c * kChunk + 64 * j, 0, h);
                    nc = c + 1;
                }
            }
            // drain: the last load of every ring slot and W_o buffer has landed
            // (a ring stage whose gathering threads gave up before issuing it
            // never completes; its wait then runs out the full bound)
            for (int kb = max(0, issued - kStages); kb < issued; ++kb)
                drain_phase(smem_u32(&sm.full[kb % kStages]), (kb / kStages) & 1);
            for (int c = max(0, nc - 2); c < nc; ++c) drain_phase(smem_u32(&sm.wo_full[c & 1]), (c >> 1) & 1);
        }
    } else if (warp == 1) {
        // ------------------------------------------------------------- MMA
        if (lane == 0) {
            bool ok = true;
            // phase 1: [Q|K|V] into TMEM columns 0..191
            constexpr uint32_t idQKV = idesc_bf16(128, 192, false, true);
            for (int kb = 0; kb < nkb && ok; ++kb) {
                const int s = kb % kStages;
                if (!(ok = wait_or_abort(sm, sm.full[s], (kb / kStages) & 1, p.status))) break;
                tc_fence_after();
                const uint32_t a = smem_u32(slot(s)), b = a + kHalf;
#pragma unroll
                for (int j = 0; j < 4; ++j)
                    mma_bf16(tmem, smem_desc_sw128(a + j * 32, 16, 1024),
                             smem_desc_sw128(b + j * 2048, 8192, 1024), idQKV,
                             (kb > 0 || j > 0) ? 1u : 0u);
                mma_commit(smem_u32(&sm.empty[s]));
            }
            mma_commit(smem_u32(&sm.qkv_done));
            // phase 3: S = Q K^T (TMEM 0..127), then O = P V (TMEM 128..191)
            ok = ok && wait_or_abort(sm, sm.qkv_staged, 0, p.status);
            if (ok) {
                tc_fence_after();
                constexpr uint32_t idS = idesc_bf16(128, 128, false, false);
                const uint32_t qa[3] = {smem_u32(sm.q[0]), smem_u32(sm.q[0]), smem_u32(sm.q[1])};
                const uint32_t kb3[3] = {smem_u32(sm.k[0]), smem_u32(sm.k[1]), smem_u32(sm.k[0])};
#pragma unroll
                for (int t = 0; t < 3; ++t)
#pragma unroll
                    for (int kk = 0; kk < 4; ++kk)
                        mma_bf16(tmem, smem_desc_sw128(qa[t] + kk * 32, 16, 1024),
                                 smem_desc_sw128(kb3[t] + kk * 32, 16, 1024), idS,
                                 (t > 0 || kk > 0) ? 1u : 0u);
            }
            mma_commit(smem_u32(&sm.s_full));
            ok = ok && wait_or_abort(sm, sm.p_ready, 0, p.status);
            if (ok) {
                tc_fence_after();
                constexpr uint32_t idO = idesc_bf16(128, 64, false, true);
                // P (K-major over the two 64-key blocks) x V (MN-major)
#pragma unroll
                for (int t = 0; t < 3; ++t) {
                    const int ah = t == 2 ? 1 : 0, bh = t == 1 ? 1 : 0;
#pragma unroll
                    for (int kk = 0; kk < 8; ++kk)
                        mma_bf16(tmem + 128,
                                 smem_desc_sw128(smem_u32(ptile[ah][kk >> 2]) + (kk & 3) * 32, 16, 1024),
                                 smem_desc_sw128(smem_u32(sm.v[bh]) + kk * 2048, kHalf, 1024), idO,
                                 (t > 0 || kk > 0) ? 1u : 0u);
                }
            }
            mma_commit(smem_u32(&sm.o_full));
            // phase 4: Y chunk c = AR (pair, K = 64) x W_o[:, chunk], TMEM 256 (c % 2)
            ok = ok && wait_or_abort(sm, sm.ar_ready, 0, p.status);
            constexpr uint32_t idY = idesc_bf16(128, kChunk, false, true);
            for (int c = 0; c < nch && ok; ++c) {
                const int buf = c & 1;
                if (!(ok = wait_or_abort(sm, sm.wo_full[buf], (c >> 1) & 1, p.status))) break;
                if (c >= 2 && !(ok = wait_or_abort(sm, sm.out_empty[buf], ((c >> 1) - 1) & 1, p.status)))
                    break;
                tc_fence_after();
                const uint32_t wb = smem_u32(buf ? &sm.v[0][0] : &sm.k[0][0]);
#pragma unroll
                for (int half = 0; half < 2; ++half)
#pragma unroll
                    for (int j = 0; j < 4; ++j)
                        mma_bf16(tmem + 256 * buf, smem_desc_sw128(smem_u32(sm.q[half]) + j * 32, 16, 1024),
                                 smem_desc_sw128(wb + j * 2048, 8192, 1024), idY,
                                 (half > 0 || j > 0) ? 1u : 0u);
                mma_commit(smem_u32(&sm.out_full[buf]));
                mma_commit(smem_u32(&sm.wo_empty[buf]));
            }
            if (!ok) {
                // release every epilogue wait that may still be pending
                for (int i = 0; i < 2; ++i) mma_commit(smem_u32(&sm.out_full[i]));
            }
            drain_mmas(smem_u32(&sm.drained));
        }
    } else if (warp == 3) {
        // ------------------------------------------------- TMA stores
        if (lane == 0) {
            // Q, K, V pairs straight from the attention operand tiles
            bool ok = wait_or_abort(sm, sm.qkv_staged, 0, p.status);
            if (ok) {
                uint8_t(*tiles[3])[kHalf] = {sm.q, sm.k, sm.v};
                for (int j = 0; j < 3; ++j)
                    for (int hf = 0; hf < 2; ++hf)
                        tma_store_3d(&p.mOut[j], smem_u32(tiles[j][hf]), 64 * hf, b0 * p.k, h);
                bulk_commit();
            }
            bulk_wait_read0();
            mbar_arrive(smem_u32(&sm.qkv_read));   // the tiles may be overwritten
            // AR pair from the Q tile (the A operand of phase 4)
            if (ok && wait_or_abort(sm, sm.ar_ready, 0, p.status)) {
                for (int hf = 0; hf < 2; ++hf)
                    tma_store_3d(&p.mOut[3], smem_u32(sm.q[hf]), 64 * hf, b0 * p.k, h);
                bulk_commit();
            }
            bulk_wait0();
        }
    } else if (warp >= 4) {
        const int t = threadIdx.x - 128;            // 0..255
        const int q = warp & 3, ch = (warp - 4) >> 2;
        const int r = q * 32 + lane;                 // tile row of this thread
        const uint32_t lane_off = (uint32_t)(q * 32) << 16;
        const int u = r / p.k;
        const bool valid = u < p.U && b0 + u < p.B;
        const int lo = valid ? u * p.k : r + 1;     // first visible key (none when invalid)
        const size_t grow0 = row_base + q * 32;     // head row of lane 0's tile row

        // ------------------------------------------- phase 1: gather X rows
        {
            const int chunk = t & 7, sub = t >> 3;  // 32 rows x 8 chunks per pass
            int landed = 0, issued = 0;
            for (int kb = 0; kb < nkb; ++kb) {
                const int s = kb % kStages;
                if (!wait_or_abort(sm, sm.empty[s], ((kb / kStages) & 1) ^ 1, p.status)) break;
                const uint32_t a = smem_u32(slot(s));
                const int col = kb * 64 + chunk * 8;
#pragma unroll
                for (int j = 0; j < 4; ++j) {
                    const int row = sub + 32 * j;
                    const int src = sm.rows[row];
                    const uint32_t nbytes = (src >= 0 && col < p.d) ? 16u : 0u;
                    const bf16 *g = p.X + (size_t)(src >= 0 ? src : 0) * p.d + (nbytes ? col : 0);
                    cp_async16(a + row * 128 + ((chunk ^ (row & 7)) << 4), g, nbytes);
                }
                cp_async_commit();
                issued = kb + 1;
                if (kb >= kLag) {
                    cp_async_wait<kLag>();
                    fence_proxy_async();
                    mbar_arrive(smem_u32(&sm.full[(kb - kLag) % kStages]));
                    ++landed;
                }
            }
            cp_async_wait<0>();
            fence_proxy_async();
            for (int kb = landed; kb < issued; ++kb) mbar_arrive(smem_u32(&sm.full[kb % kStages]));
        }

        // ------------------- phase 2: Q|K|V pairs into shared and global memory
        bool ok = wait_or_abort(sm, sm.qkv_done, 0, p.status);
        tc_fence_after();
        for (int c0 = 96 * ch; c0 < 96 * ch + 96; c0 += 32) {
            float v[32];
            tmem_ld32(tmem + lane_off + c0, v);
            if (p.rope_on && (c0 == 0 || c0 == 64) && valid) {
                // the first h'/2 = 32 columns of Q (c0 = 0) and of K (c0 = 64)
                const int t = sm.rows[r] % p.rope.T;
#pragma unroll
                for (int pr = 0; pr < 16; ++pr) rope_turn(v[2 * pr], v[2 * pr + 1], p.rope.phi[pr], t, 1.f);
            }
            uint8_t(*tile)[kHalf] = c0 < 64 ? sm.q : (c0 < 128 ? sm.k : sm.v);
            put_pair32(tile[0], tile[1], r, c0, v, 1.f);
        }
        fence_proxy_async();
        tc_fence_before();
        named_barrier(1, kWorkers);
        mbar_arrive(smem_u32(&sm.qkv_staged));

        // -------------------------------------------------- phase 3: softmax
        ok = wait_or_abort(sm, sm.s_full, 0, p.status) && ok;
        tc_fence_after();
        const int cb = 64 * ch;   // this thread's 64 keys
        float m = -INFINITY;
#pragma unroll 1
        for (int c0 = cb; c0 < cb + 64; c0 += 32) {
            float t32[32];
            tmem_ld32(tmem + lane_off + c0, t32);
#pragma unroll
            for (int c = 0; c < 32; ++c)
                if (c0 + c <= r && c0 + c >= lo) m = fmaxf(m, t32[c] * p.scale_log2);
        }
        sm.part_max[ch][r] = m;
        named_barrier(1, kWorkers);
        m = fmaxf(sm.part_max[0][r], sm.part_max[1][r]);
        float l = 0.f;
#pragma unroll 1
        for (int c0 = cb; c0 < cb + 64; c0 += 32) {
            float t32[32];
            tmem_ld32(tmem + lane_off + c0, t32);
#pragma unroll
            for (int c = 0; c < 32; ++c) {
                t32[c] = (c0 + c <= r && c0 + c >= lo) ? exp2_fast(t32[c] * p.scale_log2 - m) : 0.f;
                l += t32[c];
            }
            put_pair32(ptile[0][c0 >> 6], ptile[1][c0 >> 6], r, c0, t32, 1.f);
        }
        sm.part_sum[ch][r] = l;
        fence_proxy_async();
        tc_fence_before();
        mbar_arrive(smem_u32(&sm.p_ready));
        ok = wait_or_abort(sm, sm.o_full, 0, p.status) && ok;
        tc_fence_after();
        named_barrier(1, kWorkers);   // partial sums visible; Q tile no longer read
        ok = wait_or_abort(sm, sm.qkv_read, 0, p.status) && ok;   // nor by its TMA store
        l = sm.part_sum[0][r] + sm.part_sum[1][r];
        float o[32];
        tmem_ld32(tmem + 128 + lane_off + 32 * ch, o);   // output columns 32 ch .. +31
        const float inv = valid ? 1.f / l : 0.f;
        const float rr = valid ? p.rsel[grow0 + lane] : 0.f;
        // AR pair into the Q tile (A operand of phase 4), columns 32 ch .. +31
        put_pair32(sm.q[0], sm.q[1], r, 32 * ch, o, inv * rr);
        fence_proxy_async();
        tc_fence_before();
        mbar_arrive(smem_u32(&sm.ar_ready));
        const bool live = __all_sync(0xffffffffu, ok && !*(volatile int *)&sm.abort);
        uint8_t *xb = stage_area + (warp - 4) * 4096;
        if (live && ch == 0 && valid) p.lse[grow0 + lane] = (m + log2f(l)) * 0.69314718055994531f;

        // ------------------------------------- phase 4: scatter-add into Y
        const int cu = lane & 7;
        for (int c = 0; c < nch; ++c) {
            const int buf = c & 1;
            const bool got = wait_or_abort(sm, sm.out_full[buf], (c >> 1) & 1, p.status);
            tc_fence_after();
            const bool go = __all_sync(0xffffffffu, got && live);
            const uint32_t tb = tmem + 256 * buf + lane_off;
#pragma unroll 1
            for (int s0 = 128 * ch; s0 < 128 * ch + 128; s0 += 32) {
                if (!go) break;
                float v[32];
                tmem_ld32(tb + s0, v);
                stage_f32x32(xb, v, 1.f, lane);
                const int n = c * kChunk + s0 + 4 * cu;
#pragma unroll
                for (int i = 0; i < 8; ++i) {
                    const int rl = (lane >> 3) + 4 * i;
                    const int src = sm.rows[q * 32 + rl];
                    const float4 val = *reinterpret_cast<const float4 *>(xb + xoff128(rl, cu));
                    if (src >= 0 && n < p.d)
                        red_add_v4(p.Y + (size_t)src * p.d + n, val.x, val.y, val.z, val.w);
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

// Per-head tiles of a [H, rows, cols] bf16 array: box {64, box_rows, 1}.
bool map_heads3(CUtensorMap *m, const void *base, uint64_t H, uint64_t rows, uint64_t cols,
                uint32_t box_rows) {
    const uint64_t dims[3] = {cols, rows, H}, strides[2] = {cols * 2, rows * cols * 2};
    const uint32_t box[3] = {64, box_rows, 1};
    return tmap_bf16(m, base, 3, dims, strides, box);
}

}  // namespace

bool tc_fused_forward_supported(const Dims &dm) { return tc_supported(dm) && dm.k <= 128; }

cudaError_t tc_fused_forward(const Dims &dm, const void *X, const void *Wq, const void *Wk,
                             const void *Wv, const void *Wo, const Saved &sv, float *Y,
                             cudaStream_t s) {
    FusedParams p;
    memset(&p, 0, sizeof(p));
    const void *W[3] = {Wq, Wk, Wv};
    const int U = 128 / dm.k;
    const void *outs[4] = {sv.Q, sv.K, sv.V, sv.AR};
    bool ok = map_heads3(&p.mWo, Wo, dm.H, 64, dm.d, 64);
    for (int j = 0; j < 3; ++j) ok = ok && map_heads3(&p.mW[j], W[j], dm.H, dm.d, 64, 64);
    for (int j = 0; j < 4; ++j)
        ok = ok && map_heads3(&p.mOut[j], outs[j], dm.H, (uint64_t)dm.B * dm.k, 128, U * dm.k);
    if (!ok) return cudaErrorInvalidValue;
    p.X = static_cast<const bf16 *>(X);
    p.gidx = sv.gidx;
    p.rsel = sv.rsel;
    p.lse = sv.lse;
    p.Y = Y;
    p.B = dm.B;
    p.T = dm.T;
    p.d = dm.d;
    p.k = dm.k;
    p.U = 128 / dm.k;
    p.Mtok = dm.B * dm.k;
    p.scale_log2 = 1.4426950408889634f / sqrtf(64.f);
    p.rope_on = dm.rope ? 1 : 0;
    if (dm.rope) p.rope = make_rope_table(64, dm.T);
    p.status = sv.status;
    p.span = active_span();
    const cudaError_t attr = allow_smem((const void *)fused_fwd_kernel, kSmem);
    if (attr != cudaSuccess) return attr;
    const dim3 grid((dm.B + p.U - 1) / p.U, dm.H);
    cudaError_t e = launch_pdl(fused_fwd_kernel, grid, dim3(kThreads), kSmem, s, p);
    note_launches(1);
    return e;
}

}  // namespace mosa
