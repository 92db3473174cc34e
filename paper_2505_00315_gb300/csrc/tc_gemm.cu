// Per-head projections of the MoSA layer on the 5th-generation tensor cores
// (tcgen05.mma, fp32 accumulators in TMEM): dense operands staged by TMA, the
// rows gathered through the selected token indices by 16-byte cp.async copies.
//
// One CTA computes one 128-row output tile of one head (or one split of the
// reduction for the weight gradients).  Warp roles (256 threads):
//   warp 0      producer: TMA tile loads into a STAGES-deep ring
//   warp 1      MMA issuer (one thread): tcgen05.mma per 16-wide K step
//   warp 2      TMEM allocator
//   warps 4-7   gathered operand: 16-byte cp.async copies of the selected rows,
//               written in the 128-byte-swizzled layout (TMA gather4 issues
//               only ~4 rows per ~80 cycles per SM, too slow here); then the
//               epilogue: tcgen05.ld of the accumulator rows and the fused
//               output step of each variant.  Wide tiles (kQKV, kDWO, kDW,
//               kROUTER) split the epilogue over all eight warps, two per TMEM
//               lane quadrant, each taking half of the columns.
// Every mbarrier wait is bounded; a wait that runs out sets kStatusTimeout in
// the workspace status word and the CTA winds down without hanging.
//
// Variants (bf16 inputs, head size 64; intermediates are bf16 hi/lo pairs, so
// a product with one is two MMAs into the same accumulator):
//   kQKV  F3  [Q|K|V](m,:)  = X[g(m),:] W_{q|k|v}[h]        A gathered K-major, B MN-major
//   kG    B1  G(m,:)        = dY[g(m),:] W_o[h]^T, then D = <AR, G>, dA = r G, dlogit in the epilogue
//   kDWO  B1  dW_o[h](p,c)  = sum_m AR(m,p) dY[g(m),c]       A gathered MN-major, B = AR pair
//   kDW   B4  [dW_q|dW_k|dW_v|dW_r][h](c,:) = sum_m X[g(m),c] [dQ|dK|dV|dlogit](m,:)
//             A gathered MN-major, B = the dQKV pair (column 0 of its 4th 64-column
//             block holds dlogit; the rest of that block only reaches unread
//             accumulator columns), so dW_r comes out of the same product;
//             256 rows c per CTA in two accumulators that share every B tile
//   kROUTER F1 r[b,h,t] = sigmoid(X[b,t,:] W_r[:,h])       A = X tiles, B = W_r MN-major
// where g(m) = b*T + I[b,h,i] for row m = b*k + i of head h.  The products
// that scatter-add rows into Y or dX (F5 for k > 128, B3) have a persistent
// kernel of their own (tc_dx.cu).
#include <algorithm>
#include <cstdio>
#include <cstdlib>
#include <mutex>

#include "launch.h"
#include "profile.h"
#include "tc_common.cuh"
#include "tmap.h"

namespace mosa {
namespace {

using namespace tc;

// (the values name the kernel instances tc_gemm_kernel<N> in profiles)
enum Kind : int { kQKV = 0, kG = 2, kDWO = 3, kDW = 4, kROUTER = 5, kDWH = 6 };

constexpr int kBM = 128;        // rows per tile (TMEM lanes)
constexpr int kBK = 64;         // K per stage: one 128-byte swizzle row of bf16
constexpr int kTile8K = 8192;   // one 64x64 bf16 block
constexpr int kTile16K = 16384; // one 128x64 bf16 block
constexpr int kThreads = 256;
constexpr int kMaxStages = 8;    // mbarrier slots per ring

template <int KIND>
struct Cfg;
template <>
struct Cfg<kQKV> {
    static constexpr int BN = 192, STAGES = 2, A_BYTES = kTile16K, B_BYTES = 3 * kTile8K,
                         TMEM_COLS = 256, MIN_CTAS = 2;
    static constexpr bool A_MN = false, B_MN = true, A_PAIR = false, B_PAIR = false;
};
template <>
struct Cfg<kG> {
    static constexpr int BN = 64, STAGES = 4, A_BYTES = kTile16K, B_BYTES = kTile8K,
                         TMEM_COLS = 64, MIN_CTAS = 2;
    static constexpr bool A_MN = false, B_MN = false, A_PAIR = false, B_PAIR = false;
};
template <>
struct Cfg<kDWO> {
    static constexpr int BN = 64, STAGES = 3, A_BYTES = kTile16K, B_BYTES = 2 * kTile8K,
                         TMEM_COLS = 64, MIN_CTAS = 2;
    static constexpr bool A_MN = true, B_MN = true, A_PAIR = false, B_PAIR = true;
};
template <>
struct Cfg<kDW> {
    // 256 rows of d per CTA as two 128 x 256 accumulators sharing each B tile;
    // K blocks of 32 tokens: A = 4 blocks of 32 x 64, B = 8 blocks of 32 x 64
    static constexpr int BN = 256, STAGES = 4, A_BYTES = 4 * 4096, B_BYTES = 8 * 4096,
                         TMEM_COLS = 512, MIN_CTAS = 1;
    static constexpr bool A_MN = true, B_MN = true, A_PAIR = false, B_PAIR = true;
};

template <>
struct Cfg<kDWH> {
    // kDW on the fp16 attention path: dQ|dK|dV|dlogit single fp16 (B 16 KB a
    // stage), so the ring holds six stages and the gathers of X run four
    // stages ahead (with four they ran two ahead and bound the kernel)
    static constexpr int BN = 256, STAGES = 6, A_BYTES = 4 * 4096, B_BYTES = 4 * 4096,
                         TMEM_COLS = 512, MIN_CTAS = 1;
    static constexpr bool A_MN = true, B_MN = true, A_PAIR = false, B_PAIR = false;
};

template <>
struct Cfg<kROUTER> {
    // ring of 192 KB; the stage count is chosen at launch from the MMA width
    // (p.N = 64..256): a stage holds the X tile and N/64 W_r blocks
    static constexpr int BN = 256, STAGES = 4, A_BYTES = kTile16K, B_BYTES = 4 * kTile8K,
                         TMEM_COLS = 256, MIN_CTAS = 1;
    static constexpr bool A_MN = false, B_MN = true, A_PAIR = false, B_PAIR = false;
};

// Tokens per K block and accumulators (128-row tiles) per CTA.
template <int KIND>
__host__ __device__ constexpr int kind_bk() {
    return (KIND == kDW || KIND == kDWH) ? 32 : kBK;
}
template <int KIND>
__host__ __device__ constexpr int kind_acc() {
    return (KIND == kDW || KIND == kDWH) ? 2 : 1;
}

// Row width (bf16) of the dQKV pair array on the tensor-core path:
// [dQ | dK | dV | dlogit, 0..] hi (256) then the same lo (256).
constexpr int kDQKVCols = 512;

// Kinds whose A operand is gathered through the selected rows.
template <int KIND>
__host__ __device__ constexpr bool gathers() {
    return KIND == kQKV || KIND == kG || KIND == kDWO || KIND == kDW || KIND == kDWH;
}

// Kinds whose epilogue runs on all eight warps (wide output tiles).
template <int KIND>
__host__ __device__ constexpr bool epi_all_warps() {
    return KIND == kQKV || KIND == kDW || KIND == kDWH || KIND == kDWO || KIND == kROUTER;
}

// Kinds whose gathered operand runs along the reduction (tokens of K blocks):
// their row indices are staged in shared memory for the CTA's whole K range
// when it holds at most kIdxMax tokens (each K block otherwise began with a
// dependent global load of its indices, about one memory latency per block).
template <int KIND>
__host__ __device__ constexpr bool stages_idx() {
    return KIND == kDWO || KIND == kDW || KIND == kDWH;
}
constexpr int kIdxMax = 2048;

template <int KIND>
constexpr int smem_bytes() {
    return 1024 /* alignment slack */ + Cfg<KIND>::STAGES * (Cfg<KIND>::A_BYTES + Cfg<KIND>::B_BYTES) +
           2048 /* barriers, row indices, row scalars */ +
           (stages_idx<KIND>() ? kIdxMax * 4 : 0) /* K-range row indices */;
}

struct TcParams {
    CUtensorMap mapA;      // gathered source (2-D, box 64x1) or per-head tile map (3-D)
    CUtensorMap mapB[3];   // per-head tile maps of the B operand
    int M;                 // output rows per head: B*k for row kinds, d for kDWO / kDW
    int Mtok;              // selected rows per head, B*k
    int N;                 // MMA width (kROUTER)
    int ring_stages;       // kROUTER: stages in the ring (<= kMaxStages)
    int ring_stride;       // kROUTER: bytes per stage
    int nkb;               // K blocks in the whole reduction
    int splits;            // reduction splits (kDWO / kDW)
    int d, H, T;
    const int32_t *gidx;   // [H, B*k]
    const float *rsel;     // [H, B*k]
    const bf16 *ARp;       // [H, B*k, 128] pair of AR = diag(r) A (kG)
    const void *src_rows;  // gathered source [B*T, d] bf16: X (kQKV, kDW) or dY (kG, kDWO)
    void *out[3];          // Q/K/V pairs (kQKV); dA pair, dQKV pair (kG)
    float *out_f;          // r (kROUTER), dW_o (kDWO), dW_q (kDW)
    float *out_f1;         // Dd (kG), dW_k (kDW)
    float *out_f2;         // dlogit (kG), dW_v (kDW)
    float *out_f3;         // dW_r (kDW)
    uint32_t *status;
    int half;              // kQKV / kG: Q, K, V or dA as fp16 rows [H, B*k, 64] (k > 128)
                           // instead of bf16 pairs
    int dq16;              // kG: dlogit into fp16 dQ|dK|dV|dlogit rows [H, B*k, 256]
    int rope;              // kQKV with half: rotate Q and K (Sec. 2.2) before rounding
    RopeTable rope_tab;
    unsigned long long *span;   // measurement: this stage's kernel span slot, or null
    float *zero_rows;      // kG: [H, B*k, 64] fp32 rows zeroed alongside (the dQ
                           // accumulator of the k > 128 attention backward), or null
    unsigned long long wait_ns; // limit of each main-loop wait (the waits that let
                                // copies and MMAs in flight finish keep kWaitLimitNs)
};

// Epilogue staging: each warp owns kXpose bytes at the start of the operand
// ring (free once the last MMA has completed).
constexpr int kXpose = 8192;

// Byte offset of 16-byte unit u (0..15) of row rl (0..31) in a warp's 32 x 256-byte
// staging buffer.  The XOR keeps both the row-per-lane writes and the
// unit-per-lane reads free of shared-memory bank conflicts.
__device__ __forceinline__ uint32_t xoff256(int rl, int u) {
    return (uint32_t)(rl * 256 + ((u ^ (rl & 15)) << 4));
}

// Values v[8u .. 8u+7] of this lane's row as hi unit u and lo unit 8 + u.
__device__ __forceinline__ void stage_pair_unit(uint8_t *xb, int lane, int u, const float *v) {
    uint32_t h4[4], l4[4];
#pragma unroll
    for (int e = 0; e < 4; ++e) {
        split_pair2(v[2 * e], v[2 * e + 1], h4[e], l4[e]);
    }
    *reinterpret_cast<uint4 *>(xb + xoff256(lane, u)) = make_uint4(h4[0], h4[1], h4[2], h4[3]);
    *reinterpret_cast<uint4 *>(xb + xoff256(lane, 8 + u)) = make_uint4(l4[0], l4[1], l4[2], l4[3]);
}

// This lane's 64 values as one bf16 pair row [hi 0..63 | lo 0..63] of the staging buffer.
__device__ __forceinline__ void stage_pair_vals64(uint8_t *xb, const float (&v)[64], int lane) {
#pragma unroll
    for (int u = 0; u < 8; ++u) stage_pair_unit(xb, lane, u, v + 8 * u);
    __syncwarp();
}

// TMEM columns taddr .. taddr+63 of this lane's row as one bf16 pair row.
__device__ __forceinline__ void stage_pair_row64(uint8_t *xb, uint32_t taddr, int lane) {
#pragma unroll
    for (int hlf = 0; hlf < 2; ++hlf) {
        float v[32];
        tmem_ld32(taddr + 32 * hlf, v);
#pragma unroll
        for (int u = 0; u < 4; ++u) stage_pair_unit(xb, lane, 4 * hlf + u, v + 8 * u);
    }
    __syncwarp();
}

// This lane's 64 values as one fp16 row (128 bytes: units 0..7 at
// xoff128(lane, u)); returns the largest magnitude (fp16 range check).
__device__ __forceinline__ float stage_f16_vals64(uint8_t *xb, const float (&v)[64], int lane) {
    float mx = 0.f;
#pragma unroll
    for (int u = 0; u < 8; ++u) {
        uint32_t w[4];
#pragma unroll
        for (int e = 0; e < 4; ++e) {
            const float a = v[8 * u + 2 * e], b = v[8 * u + 2 * e + 1];
            mx = fmaxf(mx, fmaxf(fabsf(a), fabsf(b)));
            w[e] = pack_f16x2(a, b);
        }
        *reinterpret_cast<uint4 *>(xb + xoff128(lane, u)) = make_uint4(w[0], w[1], w[2], w[3]);
    }
    __syncwarp();
    return mx;
}

// The warp's 32 256-byte bf16 pair rows of AR into the staging buffer (unit u
// of row rl at xoff256(rl, u)), 16 lanes per row so that every load
// instruction reads two whole rows, all sixteen loads in flight before the
// first store; src_row(rl) gives the source row or nullptr to leave that
// staging row unwritten.  Each lane then reads its own row back with
// ld_staged_pair.  (One lane per row, each load instruction touched 32 rows.)
template <typename F>
__device__ __forceinline__ void load_rows256(uint8_t *xb, int lane, F src_row) {
    const int u = lane & 15;
    uint4 v[16];
#pragma unroll
    for (int i = 0; i < 16; ++i) {
        const uint4 *src = src_row((lane >> 4) + 2 * i);
        v[i] = src != nullptr ? src[u] : make_uint4(0u, 0u, 0u, 0u);
    }
#pragma unroll
    for (int i = 0; i < 16; ++i)
        *reinterpret_cast<uint4 *>(xb + xoff256((lane >> 4) + 2 * i, u)) = v[i];
    __syncwarp();
}

// This lane's staged pair row: hi units 0..7, lo units 8..15 (zeros if !live).
__device__ __forceinline__ void ld_staged_pair(const uint8_t *xb, int lane, bool live, uint4 (&ah)[8],
                                               uint4 (&al)[8]) {
#pragma unroll
    for (int u = 0; u < 8; ++u) {
        ah[u] = live ? *reinterpret_cast<const uint4 *>(xb + xoff256(lane, u)) : make_uint4(0u, 0u, 0u, 0u);
        al[u] = live ? *reinterpret_cast<const uint4 *>(xb + xoff256(lane, 8 + u)) : make_uint4(0u, 0u, 0u, 0u);
    }
    __syncwarp();
}

// Copies staged rows 0 .. nrows-1 to global memory with 16 lanes per row, so
// every store instruction writes two whole 256-byte rows; addr(rl, u) gives
// the destination of unit u of row rl.
template <typename F>
__device__ __forceinline__ void store_rows256(const uint8_t *xb, int lane, int nrows, F addr) {
    const int u = lane & 15;
#pragma unroll 4
    for (int i = 0; i < 16; ++i) {
        const int rl = (lane >> 4) + 2 * i;
        const uint4 val = *reinterpret_cast<const uint4 *>(xb + xoff256(rl, u));
        if (rl < nrows) *addr(rl, u) = val;
    }
    __syncwarp();
}

// TMEM columns taddr .. taddr+31 of this lane's row into a 32 x 128-byte
// buffer: 16-byte unit c of row rl at rl*128 + ((c ^ (rl & 7)) << 4).
__device__ __forceinline__ void stage_f32_32(uint8_t *xb, uint32_t taddr, int lane) {
    float v[32];
    tmem_ld32(taddr, v);
#pragma unroll
    for (int c = 0; c < 8; ++c)
        *reinterpret_cast<float4 *>(xb + lane * 128 + ((c ^ (lane & 7)) << 4)) =
            make_float4(v[4 * c], v[4 * c + 1], v[4 * c + 2], v[4 * c + 3]);
    __syncwarp();
}

// The gathered A operand of one stage, copied by the 128 threads of warps 4-7
// with 16-byte cp.async into the 128-byte-swizzled layout the MMA reads:
//   K-major (kQKV, kG):    rows m of the tile = source rows g(m), 64 columns of K block kb
//   MN-major (kDWO):       64 tokens of K block kb, columns m0 .. m0+127 in two
//                          64-wide blocks; token rows are the smem rows
//   MN-major (kDW):        32 tokens of K block kb, columns m0 .. m0+255 in four
//                          64-wide blocks
// Element (row, 16-byte chunk c) lands at row*128 + ((c ^ (row & 7)) * 16).
// A stage's copies are confirmed (wait, proxy fence, arrival on its full
// barrier) LAG stages after they are issued, with LAG = STAGES - 2 (deeper
// rings; a two-stage ring keeps LAG = 1): issuing
// stage it + LAG waits only for the MMAs of stage it - 2, so the barrier of
// stage it opens while the MMAs of stage it - 1 still run and the tensor pipe
// never drains between K blocks.
template <int KIND>
__device__ __forceinline__ void gather_operand(const TcParams &p, uint8_t *sA, uint64_t *full,
                                               uint64_t *empty, const int *s_rows, int *s_abort,
                                               int h, int m0, int kb_begin, int nkb,
                                               const int *s_idx, int tok0, bool idx_staged) {
    using C = Cfg<KIND>;
    constexpr int S = C::STAGES;
    constexpr int LAG = S >= 3 ? S - 2 : S - 1;  // a two-stage ring keeps one stage of lag
    const int t = threadIdx.x - 128;       // 0..127
    const int chunk = t & 7, sub = t >> 3;  // 16 rows x 8 chunks per pass
    const bf16 *src = static_cast<const bf16 *>(p.src_rows);
    const int32_t *gi = p.gidx + (size_t)h * p.Mtok;
    int landed = 0;  // stages whose full barrier this thread has arrived on
    int issued = 0;  // stages whose copies this thread has issued
    for (int it = 0; it < nkb; ++it) {
        const int s = it % S;
        if (!mbar_wait(smem_u32(&empty[s]), ((it / S) & 1) ^ 1, p.wait_ns) ||
            *(volatile int *)s_abort) {
            atomicOr(p.status, kStatusTimeout);
            *(volatile int *)s_abort = 1;
            break;
        }
        const int kb = kb_begin + it;
        const uint32_t a = smem_u32(sA + s * C::A_BYTES);
        if constexpr (KIND == kQKV || KIND == kG) {
            const int col = kb * kBK + chunk * 8;
            const uint32_t nbytes = col < p.d ? 16u : 0u;
#pragma unroll
            for (int j = 0; j < 8; ++j) {
                const int row = sub + 16 * j;
                const bf16 *g = src + (size_t)s_rows[row] * p.d + (nbytes ? col : 0);
                cp_async16(a + row * 128 + ((chunk ^ (row & 7)) << 4), g, nbytes);
            }
        } else if constexpr (KIND == kDW || KIND == kDWH) {
            // 32 tokens x 256 columns of d in four 64-wide blocks of 4 KB
#pragma unroll
            for (int q2 = 0; q2 < 2; ++q2) {
                const int tok = sub + 16 * q2;
                const int tg = kb * 32 + tok;
                const int rowg = idx_staged ? s_idx[tg - tok0] : (tg < p.Mtok ? gi[tg] : 0);
#pragma unroll
                for (int j = 0; j < 4; ++j) {
                    const int col = m0 + 64 * j + chunk * 8;
                    const uint32_t nbytes = (tg < p.Mtok && col < p.d) ? 16u : 0u;
                    const bf16 *g = src + (size_t)rowg * p.d + (nbytes ? col : 0);
                    cp_async16(a + j * 4096 + tok * 128 + ((chunk ^ (tok & 7)) << 4), g, nbytes);
                }
            }
        } else {
#pragma unroll
            for (int q4 = 0; q4 < 4; ++q4) {
                const int tok = sub + 16 * q4;
                const int tg = kb * kBK + tok;
                const int rowg = idx_staged ? s_idx[tg - tok0] : (tg < p.Mtok ? gi[tg] : 0);
#pragma unroll
                for (int j = 0; j < 2; ++j) {
                    const int col = m0 + 64 * j + chunk * 8;
                    const uint32_t nbytes = (tg < p.Mtok && col < p.d) ? 16u : 0u;
                    const bf16 *g = src + (size_t)rowg * p.d + (nbytes ? col : 0);
                    cp_async16(a + j * kTile8K + tok * 128 + ((chunk ^ (tok & 7)) << 4), g, nbytes);
                }
            }
        }
        cp_async_commit();
        issued = it + 1;
        if (it >= LAG) {
            cp_async_wait<LAG>();
            fence_proxy_async();
            mbar_arrive(smem_u32(&full[(it - LAG) % S]));
            ++landed;
        }
    }
    // Every stage issued lands before its barrier is arrived on, also after a
    // give-up, so that the producer's drain of the same stages completes.
    cp_async_wait<0>();
    fence_proxy_async();
    for (int it = landed; it < issued; ++it) mbar_arrive(smem_u32(&full[it % S]));
}

template <int KIND>
__global__ void __launch_bounds__(kThreads, Cfg<KIND>::MIN_CTAS)
    tc_gemm_kernel(const __grid_constant__ TcParams p) {
    using C = Cfg<KIND>;
    constexpr int S = C::STAGES;
    extern __shared__ uint8_t smem_raw[];
    uint8_t *smem = reinterpret_cast<uint8_t *>(
        (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    uint8_t *sA = smem;
    uint8_t *sB = smem + S * C::A_BYTES;
    uint64_t *bars = reinterpret_cast<uint64_t *>(sB + S * C::B_BYTES);
    uint64_t *full = bars, *empty = bars + kMaxStages, *done = bars + 2 * kMaxStages;
    static_assert(S <= kMaxStages, "ring too deep");
    // the router's ring is laid out per stage ([X tile | W_r blocks]) with a
    // stage count fixed at launch; every other kind has STAGES A tiles, then
    // STAGES B tiles
    const int ns = KIND == kROUTER ? p.ring_stages : S;
    auto stage_a = [&](int st) -> uint8_t * {
        return KIND == kROUTER ? smem + st * p.ring_stride : sA + st * C::A_BYTES;
    };
    auto stage_b = [&](int st) -> uint8_t * {
        return KIND == kROUTER ? smem + st * p.ring_stride + C::A_BYTES : sB + st * C::B_BYTES;
    };
    uint32_t *tmem_slot = reinterpret_cast<uint32_t *>(done + 1);
    int *s_abort = reinterpret_cast<int *>(tmem_slot + 1);
    int *s_rows = s_abort + 1 + 2;  // 128 gather rows, 16-byte aligned below
    s_rows = reinterpret_cast<int *>((reinterpret_cast<uintptr_t>(s_rows) + 15) & ~uintptr_t(15));
    int *s_idx = s_rows + 128;      // stages_idx kinds: row indices of the CTA's K range
    static_assert(KIND == kROUTER || S * (C::A_BYTES + C::B_BYTES) >= 8 * kXpose,
                  "epilogue staging must fit in the operand ring");

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int m_tile = blockIdx.x, n_tile = blockIdx.y;
    constexpr bool kSplitK = KIND == kDWO || KIND == kDW || KIND == kDWH;
    const int h = kSplitK ? blockIdx.z / p.splits : blockIdx.z;
    const int split = kSplitK ? blockIdx.z % p.splits : 0;
    const int m0 = m_tile * kBM * kind_acc<KIND>();
    const int n0 = n_tile * C::BN;
    int kb_begin = 0, kb_end = p.nkb;
    if (kSplitK) {
        const int per = (p.nkb + p.splits - 1) / p.splits;
        kb_begin = split * per;
        kb_end = min(p.nkb, kb_begin + per);
    }
    const int nkb = kb_end - kb_begin;

    if (threadIdx.x == 0) {
        for (int s = 0; s < ns; ++s) {
            // gathered kinds: the TMA arrival plus one per gathering thread
            mbar_init(smem_u32(&full[s]), gathers<KIND>() ? 129 : 1);
            mbar_init(smem_u32(&empty[s]), 1);
        }
        mbar_init(smem_u32(done), 1);
        *s_abort = 0;
        fence_barrier_init();
    }
    pdl_wait();  // everything below may read what the previous kernel wrote
    span_begin(p.span);
    if (KIND == kQKV || KIND == kG) {
        for (int r = threadIdx.x; r < kBM; r += kThreads) {
            const int m = m0 + r;
            s_rows[r] = m < p.Mtok ? p.gidx[(size_t)h * p.Mtok + m] : 0;
        }
    }
    const int tok0 = kb_begin * kind_bk<KIND>();
    const bool idx_staged = stages_idx<KIND>() && nkb * kind_bk<KIND>() <= kIdxMax;
    if (idx_staged) {
        for (int i = threadIdx.x; i < nkb * kind_bk<KIND>(); i += kThreads) {
            const int tg = tok0 + i;
            s_idx[i] = tg < p.Mtok ? p.gidx[(size_t)h * p.Mtok + tg] : 0;
        }
    }
    if (warp == 2) {
        tmem_alloc(smem_u32(tmem_slot), C::TMEM_COLS);
        tmem_relinquish();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = *tmem_slot;

    if (warp == 0) {
        // ------------------------------------------------------- producer
        const int nbl = KIND == kROUTER ? p.N / 64 : 0;  // router: 64-wide W_r blocks per stage
        int issued = 0;
        for (int it = 0; it < nkb; ++it) {
            const int s = it % ns;
            const uint32_t fb = smem_u32(&full[s]);
            bool ok = true;
            if (lane == 0) ok = mbar_wait(smem_u32(&empty[s]), ((it / ns) & 1) ^ 1, p.wait_ns);
            ok = __shfl_sync(0xffffffffu, ok ? 1 : 0, 0) != 0;
            if (!ok || *(volatile int *)s_abort) {
                if (lane == 0) {
                    atomicOr(p.status, kStatusTimeout);
                    *(volatile int *)s_abort = 1;
                }
                break;
            }
            const int kb = kb_begin + it;
            const uint32_t a = smem_u32(stage_a(s)), b = smem_u32(stage_b(s));
            if (lane == 0) {
                const uint32_t tx = KIND == kROUTER ? C::A_BYTES + nbl * kTile8K
                                    : gathers<KIND>() ? C::B_BYTES : C::A_BYTES + C::B_BYTES;
                mbar_expect_tx(fb, tx);
            }
            __syncwarp();
            if constexpr (KIND == kQKV) {
                if (lane < 3) tma_load_3d(b + lane * kTile8K, &p.mapB[lane], fb, 0, kb * kBK, h);
            } else if constexpr (KIND == kG) {
                if (lane == 0) tma_load_3d(b, &p.mapB[0], fb, kb * kBK, 0, h);
            } else if constexpr (KIND == kROUTER) {
                if (lane == 0) tma_load_2d(a, &p.mapA, fb, kb * kBK, m0);
                if (lane >= 1 && lane <= nbl)
                    tma_load_2d(b + (lane - 1) * kTile8K, &p.mapB[0], fb, n0 + 64 * (lane - 1), kb * kBK);
            } else if constexpr (KIND == kDWO) {
                if (lane < 2) tma_load_3d(b + lane * kTile8K, &p.mapB[0], fb, 64 * lane, kb * kBK, h);
            } else if constexpr (KIND == kDWH) {  // fp16 blocks 0..3, 32 token rows each
                if (lane < 4) tma_load_3d(b + lane * 4096, &p.mapB[0], fb, 64 * lane, kb * 32, h);
            } else {  // kDW: hi blocks 0..3 then lo blocks 0..3, 32 token rows each
                if (lane < 8) tma_load_3d(b + lane * 4096, &p.mapB[0], fb, 64 * lane, kb * 32, h);
            }
            issued = it + 1;
        }
        if (lane == 0) {
            // Copies in flight land before the CTA can exit: the last load of
            // every ring slot (on the normal path all of them have been consumed).
            // For gathered kinds a stage whose gathering threads gave up before
            // issuing it never completes; its wait then runs out the full bound.
            for (int it = max(0, issued - ns); it < issued; ++it)
                drain_phase(smem_u32(&full[it % ns]), (it / ns) & 1);
        }
    } else if (warp == 1) {
        // ------------------------------------------------------ MMA issuer
        if (lane == 0) {
            const uint32_t idesc = KIND == kROUTER ? idesc_bf16(kBM, p.N, false, true)
                                   : KIND == kDWH ? idesc_f16(kBM, C::BN, C::A_MN, C::B_MN)
                                   : idesc_bf16(kBM, C::BN, C::A_MN, C::B_MN);
            for (int it = 0; it < nkb; ++it) {
                const int s = it % ns;
                if (!mbar_wait(smem_u32(&full[s]), (it / ns) & 1, p.wait_ns) ||
                    *(volatile int *)s_abort) {
                    atomicOr(p.status, kStatusTimeout);
                    *(volatile int *)s_abort = 1;
                    break;
                }
                tc_fence_after();
                const uint32_t a = smem_u32(stage_a(s)), b = smem_u32(stage_b(s));
                constexpr int pairs = (C::A_PAIR || C::B_PAIR) ? 2 : 1;
                if constexpr (KIND == kDW || KIND == kDWH) {
                    // accumulator c: rows of d-blocks 2c, 2c+1; B pair halves at +0 / +16 KB
                    // (kDWH: one fp16 B block set)
                    constexpr int halves = KIND == kDWH ? 1 : 2;
#pragma unroll
                    for (int c = 0; c < 2; ++c)
#pragma unroll
                        for (int half = 0; half < halves; ++half)
#pragma unroll
                            for (int j = 0; j < 2; ++j)
                                mma_bf16(tmem + 256 * c,
                                         smem_desc_sw128(a + c * 8192 + j * 2048, 4096, 1024),
                                         smem_desc_sw128(b + half * 16384 + j * 2048, 4096, 1024),
                                         idesc, (it > 0 || half > 0 || j > 0) ? 1u : 0u);
                } else
#pragma unroll
                for (int half = 0; half < pairs; ++half) {
                    const uint32_t ah = a + (C::A_PAIR ? half * (C::A_BYTES / 2) : 0);
                    const uint32_t bh = b + (C::B_PAIR ? half * (C::B_BYTES / 2) : 0);
#pragma unroll
                    for (int j = 0; j < kBK / 16; ++j) {
                        const uint64_t ad = C::A_MN ? smem_desc_sw128(ah + j * 2048, kTile8K, 1024)
                                                    : smem_desc_sw128(ah + j * 32, 16, 1024);
                        const uint64_t bd = C::B_MN ? smem_desc_sw128(bh + j * 2048, kTile8K, 1024)
                                                    : smem_desc_sw128(bh + j * 32, 16, 1024);
                        mma_bf16(tmem, ad, bd, idesc, (it > 0 || half > 0 || j > 0) ? 1u : 0u);
                    }
                }
                mma_commit(smem_u32(&empty[s]));
            }
            mma_commit(smem_u32(done));
        }
    } else if (warp >= 4) {
        if constexpr (gathers<KIND>()) gather_operand<KIND>(p, sA, full, empty, s_rows, s_abort, h, m0,
                                                            kb_begin, nkb, s_idx, tok0, idx_staged);
    }

    // ------------------------------------------------------------ epilogue
    // Warps 4-7 always; warps 0-3 too for the kinds with wide tiles.  Warp w
    // reads TMEM lanes 32 (w % 4) .. +31, i.e. tile rows q*32 .. q*32+31, and
    // takes column part (w < 4).  Its staging buffer for coalescing the global
    // writes lies in the operand ring, which is idle once every MMA is done.
    if (warp >= 4 || epi_all_warps<KIND>()) {
        __syncwarp();
        const int q = warp & 3;
        const int part = warp < 4 ? 1 : 0;
        const int r = q * 32 + lane;
        const int mg = m0 + r;
        const bool ok = mbar_wait(smem_u32(done), 0, p.wait_ns);
        if (!ok) {
            // Give up: stop the producer and the MMA issuer, then wait (full
            // bound) for the MMAs already issued, which the issuer's last
            // commit covers, before TMEM can be freed.
            *(volatile int *)s_abort = 1;
            mbar_wait(smem_u32(done), 0, kWaitLimitNs);
        }
        tc_fence_after();
        if (warp >= 4) pdl_trigger();  // main loop done: the next kernel may start its prologue
        // warp-uniform, since the TMEM loads below are warp-collective
        const bool abort = __any_sync(0xffffffffu, !ok || *(volatile int *)s_abort || nkb <= 0);
        if (!ok) atomicOr(p.status, kStatusTimeout);
        const uint32_t tb = tmem + ((uint32_t)(q * 32) << 16);
        uint8_t *xb = smem + warp * kXpose;
        if (abort) {
            // nothing to write
        } else if constexpr (KIND == kQKV) {
            // Q and K by warps 4-7, V by warps 0-3; one 256-byte pair row per
            // matrix row, or (half) one 128-byte fp16 row, Q and K turned by
            // RoPE first when asked
            const int nrows = min(32, p.M - (m0 + q * 32));
            float mx = 0.f;
            for (int j = part == 0 ? 0 : 2; j < (part == 0 ? 2 : 3); ++j) {
                if (!p.half) {
                    stage_pair_row64(xb, tb + 64 * j, lane);
                    bf16 *dst = static_cast<bf16 *>(p.out[j]) + ((size_t)h * p.Mtok + m0 + q * 32) * 128;
                    store_rows256(xb, lane, nrows, [&](int rl, int u) {
                        return reinterpret_cast<uint4 *>(dst + (size_t)rl * 128) + u;
                    });
                    continue;
                }
                float v[64];
                {
                    float t32[32];
                    tmem_ld32(tb + 64 * j, t32);
#pragma unroll
                    for (int c = 0; c < 32; ++c) v[c] = t32[c];
                    tmem_ld32(tb + 64 * j + 32, t32);
#pragma unroll
                    for (int c = 0; c < 32; ++c) v[32 + c] = t32[c];
                }
                if (p.rope && j < 2) {
                    // pairs (2p, 2p+1), p < 16, of the first 32 columns, at the
                    // token's original position t (gidx = b*T + t)
                    const int t = s_rows[r] % p.T;
#pragma unroll
                    for (int pp = 0; pp < 16; ++pp)
                        rope_turn(v[2 * pp], v[2 * pp + 1], p.rope_tab.phi[pp], t, 1.f);
                }
                mx = fmaxf(mx, stage_f16_vals64(xb, v, lane));
                bf16 *dst = static_cast<bf16 *>(p.out[j]) + ((size_t)h * p.Mtok + m0 + q * 32) * 64;
                store_rows128(xb, lane, [&](int rl, int c) -> uint4 * {
                    return rl < nrows ? reinterpret_cast<uint4 *>(dst + (size_t)rl * 64) + c : nullptr;
                });
            }
            if (!(mx < kF16Overflow) && mg < p.M) atomicOr(p.status, kStatusRange);
        } else if constexpr (KIND == kG) {
            // G row in two 32-column halves: D = <AR, G> = r <A, G> accumulates,
            // dA = r G is staged
            const bool live = mg < p.M;
            const size_t row = (size_t)h * p.Mtok + (live ? mg : 0);
            const float rr = live ? p.rsel[row] : 0.f;
            // the warp's 32 AR pair rows (one contiguous block), two rows per load instruction
            {
                const size_t arow0 = (size_t)h * p.Mtok + m0 + q * 32;
                load_rows256(xb, lane, [&](int rl) -> const uint4 * {
                    return m0 + q * 32 + rl < p.M ? reinterpret_cast<const uint4 *>(p.ARp + (arow0 + rl) * 128)
                                                  : nullptr;
                });
            }
            uint4 ah[8], al[8];
            ld_staged_pair(xb, lane, live, ah, al);
            float dd = 0.f, amax = 0.f;
#pragma unroll
            for (int hlf = 0; hlf < 2; ++hlf) {
                float g[32];
                tmem_ld32(tb + 32 * hlf, g);
#pragma unroll
                for (int u = 0; u < 4; ++u) dd = dot_pair8(ah[4 * hlf + u], al[4 * hlf + u], g + 8 * u, dd);
#pragma unroll
                for (int e = 0; e < 32; ++e) g[e] *= rr;  // dA = r G
                if (!p.half) {
#pragma unroll
                    for (int u = 0; u < 4; ++u) stage_pair_unit(xb, lane, 4 * hlf + u, g + 8 * u);
                } else {
                    // fp16 row: units 4 hlf .. 4 hlf + 3 of the 128-byte layout
#pragma unroll
                    for (int u = 0; u < 4; ++u) {
                        uint32_t w[4];
#pragma unroll
                        for (int e = 0; e < 4; ++e) {
                            const float a = g[8 * u + 2 * e], b = g[8 * u + 2 * e + 1];
                            amax = fmaxf(amax, fmaxf(fabsf(a), fabsf(b)));
                            w[e] = pack_f16x2(a, b);
                        }
                        *reinterpret_cast<uint4 *>(xb + xoff128(lane, 4 * hlf + u)) =
                            make_uint4(w[0], w[1], w[2], w[3]);
                    }
                }
            }
            __syncwarp();
            // D = rowsum(dA o A) = r <A, G>; dlogit = r (1 - r) <A, G> = D (1 - r)
            const float dl = dd * (1.f - rr);
            if (live) {
                p.out_f1[row] = dd;
                p.out_f2[row] = dl;
            }
            const int row0 = m0 + q * 32;
            const int nrows = min(32, p.M - row0);
            if (p.zero_rows != nullptr && nrows > 0) {
                // this warp's rows of the dQ accumulator: one contiguous block
                float4 *z = reinterpret_cast<float4 *>(p.zero_rows + ((size_t)h * p.Mtok + row0) * 64);
                for (int u = lane; u < nrows * 16; u += 32) z[u] = make_float4(0.f, 0.f, 0.f, 0.f);
            }
            if (!p.half) {
                bf16 *dA = static_cast<bf16 *>(p.out[0]) + ((size_t)h * p.Mtok + row0) * 128;
                store_rows256(xb, lane, nrows, [&](int rl, int u) {
                    return reinterpret_cast<uint4 *>(dA + (size_t)rl * 128) + u;
                });
            } else {
                bf16 *dA = static_cast<bf16 *>(p.out[0]) + ((size_t)h * p.Mtok + row0) * 64;
                store_rows128(xb, lane, [&](int rl, int c) -> uint4 * {
                    return rl < nrows ? reinterpret_cast<uint4 *>(dA + (size_t)rl * 64) + c : nullptr;
                });
                if (!(amax < kF16Overflow) && live) atomicOr(p.status, kStatusRange);
            }
            // dlogit as column 192 (hi) / 448 (lo) of the dQKV pair row, column 0 of
            // the 4th 64-column block that kDW reads for dW_r; the block's other
            // columns are never written: accumulator column n of that product
            // depends only on B column n, and columns 193..255 are not read
            if (live && !p.dq16) {
                const bf16 dh = __float2bfloat16_rn(dl);
                const bf16 dlo = __float2bfloat16_rn(dl - __bfloat162float(dh));
                bf16 *dq = static_cast<bf16 *>(p.out[1]) + row * kDQKVCols;
                dq[192] = dh;
                dq[448] = dlo;
            } else if (live) {
                // fp16 rows [H, B*k, 256]: dlogit at column 192
                __half *dq = static_cast<__half *>(p.out[1]) + row * 256;
                dq[192] = __float2half_rn(dl);
                if (!(fabsf(dl) < kF16Overflow)) atomicOr(p.status, kStatusRange);
            }
        } else if constexpr (KIND == kROUTER) {
            const bool live = mg < p.M;
            const int bb = live ? mg / p.T : 0, t = live ? mg % p.T : 0;
            float *dst = p.out_f + (size_t)bb * p.H * p.T + t;
            const int ncols = min(C::BN, p.H - n0);
            // 32-column groups alternate between the two warps of a lane quarter;
            // sigmoid(x) = 1 / (1 + 2^(-x log2 e)) with the hardware exp2 and
            // approximate reciprocal (relative error a few ulp; with the
            // correctly rounded reciprocal the router took 22.5 us at
            // B4 T4096 d1024 H256, 16.3 with this)
            for (int c0 = 32 * part; c0 < ncols; c0 += 64) {
                float v[32];
                tmem_ld32(tb + c0, v);
                const int nv = live ? min(32, ncols - c0) : 0;
#pragma unroll
                for (int e = 0; e < 32; ++e) {
                    if (e < nv)
                        dst[(size_t)(n0 + c0 + e) * p.T] =
                            rcp_approx(1.f + exp2_fast(-1.4426950408889634f * v[e]));
                }
            }
        } else if constexpr (KIND == kDWO) {
            // columns p = c0 .. c0+31 of this head's dW_o rows; TMEM lane = output column mg
            const int c0 = 32 * part;
            float v[32];
            tmem_ld32(tb + c0, v);
            float *xf = reinterpret_cast<float *>(xb);
#pragma unroll
            for (int e = 0; e < 32; ++e) xf[e * 32 + lane] = v[e];
            __syncwarp();
            const int mcol = m0 + q * 32 + 4 * (lane & 7);
#pragma unroll
            for (int i = 0; i < 8; ++i) {
                const int e = (lane >> 3) + 4 * i;
                const float4 val = *reinterpret_cast<const float4 *>(xf + e * 32 + 4 * (lane & 7));
                if (mcol < p.M) {
                    float *dst = p.out_f + ((size_t)h * 64 + c0 + e) * p.d + mcol;
                    if (p.splits > 1)
                        red_add_v4(dst, val.x, val.y, val.z, val.w);
                    else
                        *reinterpret_cast<float4 *>(dst) = val;
                }
            }
        } else {  // kDW / kDWH: warps 4-7 accumulator 0 (d rows m0 ..), warps 0-3 accumulator 1 (m0+128 ..)
            const int chunk = lane & 7;
            const uint32_t ta = tb + 256 * part;
            const int mrow0 = m0 + 128 * part + q * 32;
            for (int c0 = 0; c0 < 192; c0 += 32) {
                stage_f32_32(xb, ta + c0, lane);
                float *W = c0 < 64 ? p.out_f : (c0 < 128 ? p.out_f1 : p.out_f2);
#pragma unroll
                for (int i = 0; i < 8; ++i) {
                    const int rl = (lane >> 3) + 4 * i;
                    const int mr = mrow0 + rl;
                    const float4 val = *reinterpret_cast<const float4 *>(xb + rl * 128 + ((chunk ^ (rl & 7)) << 4));
                    if (mr < p.M) {
                        float *dst = W + ((size_t)h * p.d + mr) * 64 + (c0 % 64) + 4 * chunk;
                        if (p.splits > 1)
                            red_add_v4(dst, val.x, val.y, val.z, val.w);
                        else
                            *reinterpret_cast<float4 *>(dst) = val;
                    }
                }
                __syncwarp();
            }
            float v[32];
            tmem_ld32(ta + 192, v);  // column 192: dW_r[c, h]
            const int mr = mrow0 + lane;
            if (mr < p.M) {
                float *dst = p.out_f3 + (size_t)mr * p.H + h;
                if (p.splits > 1)
                    atomicAdd(dst, v[0]);
                else
                    *dst = v[0];
            }
        }
    }
    tc_fence_before();
    __syncthreads();
    span_end(p.span);
    if (warp == 2) {
        tc_fence_after();
        tmem_dealloc(tmem, C::TMEM_COLS);
    }
}

// ------------------------------------------------------------------ host

bool make_map(CUtensorMap *m, const void *base, int rank, const uint64_t *dims,
              const uint64_t *strides, const uint32_t *box) {
    return tmap_bf16(m, base, rank, dims, strides, box);
}

// Rows of a [rows, cols] bf16 matrix fetched one row (64 columns) at a time by gather4.
bool map_gather(CUtensorMap *m, const void *base, uint64_t rows, uint64_t cols) {
    const uint64_t dims[2] = {cols, rows}, strides[1] = {cols * 2};
    const uint32_t box[2] = {64, 1};
    return make_map(m, base, 2, dims, strides, box);
}

// Per-head tiles of a [H, rows, cols] bf16 array: box {64, box_rows, 1}.
bool map_heads(CUtensorMap *m, const void *base, uint64_t H, uint64_t rows, uint64_t cols,
               uint32_t box_rows) {
    const uint64_t dims[3] = {cols, rows, H}, strides[2] = {cols * 2, rows * cols * 2};
    const uint32_t box[3] = {64, box_rows, 1};
    return make_map(m, base, 3, dims, strides, box);
}

template <int KIND>
cudaError_t launch_kind(const TcParams &p, dim3 grid, cudaStream_t s, bool early = true) {
    constexpr int smem = smem_bytes<KIND>();
    if (p.wait_ns == 0) return cudaErrorInvalidValue;  // every launcher sets a wait limit
    const cudaError_t attr = allow_smem((const void *)tc_gemm_kernel<KIND>, smem);
    if (attr != cudaSuccess) return attr;
    cudaError_t e = launch_ex(early, tc_gemm_kernel<KIND>, grid, dim3(kThreads), smem, s, p);
    note_launches(1);
    return e;
}

int splits_for(int tiles, int nkb) {
    // enough CTAs to cover the 152 SMs at least once, each with >= 2 K blocks
    int sp = 1;
    while (tiles * sp < 152 && sp * 2 <= nkb / 2) sp *= 2;
    return sp;
}

TcParams base_params(const Dims &dm, const Saved &sv) {
    TcParams p;
    memset(&p, 0, sizeof(p));
    p.Mtok = dm.B * dm.k;
    p.d = dm.d;
    p.H = dm.H;
    p.gidx = sv.gidx;
    p.rsel = sv.rsel;
    p.status = sv.status;
    p.splits = 1;
    p.span = active_span();
    p.wait_ns = tc::kWaitLimitNs;
    return p;
}

// Main-loop wait limit of the router GEMM: kWaitLimitNs, or for tests of the
// give-up path the value of MOSA_TEST_ROUTER_WAIT_NS (nanoseconds, > 0).
unsigned long long router_wait_ns() {
    const char *v = std::getenv("MOSA_TEST_ROUTER_WAIT_NS");
    if (v == nullptr || v[0] == '\0') return tc::kWaitLimitNs;
    const unsigned long long ns = std::strtoull(v, nullptr, 10);
    return ns > 0 ? ns : tc::kWaitLimitNs;
}

bool map_2d(CUtensorMap *m, const void *base, uint64_t rows, uint64_t cols, uint32_t box_rows) {
    const uint64_t dims[2] = {cols, rows}, strides[1] = {cols * 2};
    const uint32_t box[2] = {64, box_rows};
    return make_map(m, base, 2, dims, strides, box);
}

}  // namespace

bool tc_router_applies(const Dims &dm) { return dm.bf16 && dm.H % 8 == 0 && tmap_available(); }

bool tc_router(const Dims &dm, const void *X, const void *Wr, int wr_cols, float *r_full,
               uint32_t *status, cudaStream_t s, cudaError_t *err) {
    if (!tc_router_applies(dm) || wr_cols < dm.H) return false;
    TcParams p;
    memset(&p, 0, sizeof(p));
    p.M = dm.B * dm.T;
    p.nkb = (dm.d + kBK - 1) / kBK;
    p.splits = 1;
    p.d = dm.d;
    p.H = dm.H;
    p.T = dm.T;
    p.status = status;
    p.span = active_span();
    p.wait_ns = router_wait_ns();
    p.out_f = r_full;
    p.N = std::min(256, (dm.H + 63) / 64 * 64);  // MMA width: 64-wide W_r blocks
    p.ring_stride = kTile16K + p.N / 64 * kTile8K;
    p.ring_stages = std::min(kMaxStages, Cfg<kROUTER>::STAGES * (kTile16K + 4 * kTile8K) / p.ring_stride);
    if (!map_2d(&p.mapA, X, (uint64_t)dm.B * dm.T, dm.d, 128) ||
        !map_2d(&p.mapB[0], Wr, dm.d, wr_cols, 64))
        return false;
    dim3 grid((p.M + kBM - 1) / kBM, (dm.H + 255) / 256, 1);
    *err = launch_kind<kROUTER>(p, grid, s);
    return true;
}

// bf16 -> fp16, eight values per 16-byte step (bf16x8_to_f16x8); a value
// beyond the fp16 range sets kStatusRange.
__global__ void to_f16_kernel(const uint4 *__restrict__ src, uint4 *__restrict__ dst, size_t n8,
                              uint32_t *status) {
    pdl_wait();
    pdl_trigger();
    bool bad = false;
    for (size_t i = (size_t)blockIdx.x * blockDim.x + threadIdx.x; i < n8;
         i += (size_t)gridDim.x * blockDim.x)
        dst[i] = bf16x8_to_f16x8(src[i], bad);
    if (__any_sync(0xffffffffu, bad) && (threadIdx.x & 31) == 0) atomicOr(status, kStatusRange);
}

__global__ void transpose_wr_kernel(const bf16 *__restrict__ Wr, float *__restrict__ WrT, int d,
                                    int H) {
    pdl_wait();
    const int i = blockIdx.x * blockDim.x + threadIdx.x;  // element of WrT [H, d]
    if (i < d * H) {
        const int h = i / d, c = i - h * d;
        WrT[i] = __bfloat162float(Wr[(size_t)c * H + h]);
    }
}

cudaError_t tc_to_f16(const void *src, void *dst, size_t n, uint32_t *status, cudaStream_t s) {
    const size_t n8 = n / 8;
    if (n8 == 0) return cudaSuccess;
    const unsigned grid = (unsigned)std::min<size_t>((n8 + 255) / 256, 1216);
    to_f16_kernel<<<grid, 256, 0, s>>>(static_cast<const uint4 *>(src), static_cast<uint4 *>(dst),
                                       n8, status);
    note_launches(1);
    return cudaGetLastError();
}

void *wo16_of(const Dims &dm, const Saved &sv) {
    return (char *)sv.W16 + 6 * (size_t)dm.H * dm.d * dm.hp;
}

cudaError_t tc_f16_copies(const Dims &dm, const void *X, const void *Wq, const void *Wk,
                          const void *Wv, const void *Wo, const Saved &sv, cudaStream_t s) {
    const size_t nw = (size_t)dm.H * dm.d * dm.hp;
    const void *src[5] = {X, Wq, Wk, Wv, Wo};
    void *dst[5] = {sv.X16, sv.W16, (char *)sv.W16 + 2 * nw, (char *)sv.W16 + 4 * nw,
                    wo16_of(dm, sv)};
    const size_t n[5] = {(size_t)dm.B * dm.T * dm.d, nw, nw, nw, nw};   // d % 8 == 0
    for (int i = 0; i < 5; ++i) {
        if (src[i] == nullptr) continue;
        const cudaError_t e = tc_to_f16(src[i], dst[i], n[i], sv.status, s);
        if (e != cudaSuccess) return e;
    }
    return cudaSuccess;
}

cudaError_t tc_transpose_wr(const Dims &dm, const void *Wr, const Saved &sv, cudaStream_t s) {
    const int n = dm.d * dm.H;
    transpose_wr_kernel<<<(n + 255) / 256, 256, 0, s>>>(static_cast<const bf16 *>(Wr), sv.WrT,
                                                        dm.d, dm.H);
    note_launches(1);
    return cudaGetLastError();
}

bool tc_supported(const Dims &dm) {
    return dm.bf16 && dm.hp == 64 && tmap_available();
}

bool attn_f16(const Dims &dm) { return dm.k > 128 && use_tc(dm); }

bool dqkv_f16(const Dims &dm) {
    if (!use_tc(dm)) return false;
    if (dm.k > 128) return true;
    if (use_fused_backward(dm)) return false;
    // k <= 128: worth the forward's fp16 copies of X and W_q|W_k|W_v while
    // the weights' copy is at most twice X's (3 H h' <= 2 B T).  Measured:
    // 101.8 against 107.0 us at B8 T1024 d512 H16 k128, 384 against 397 at
    // B16 T1024 d1024 H64 k64, 414 against 422 at B4 T4096 d1024 H128 k128;
    // 495 against 486 at H256 k64, whose weights are three times X.
    return 3LL * dm.H * dm.hp <= 2LL * dm.B * dm.T;
}

cudaError_t tc_qkv(const Dims &dm, const void *X, const void *Wq, const void *Wk, const void *Wv,
                   const Saved &sv, cudaStream_t s) {
    TcParams p = base_params(dm, sv);
    p.M = p.Mtok;
    p.nkb = (dm.d + kBK - 1) / kBK;
    bool ok = map_gather(&p.mapA, X, (uint64_t)dm.B * dm.T, dm.d);
    const void *W[3] = {Wq, Wk, Wv};
    for (int j = 0; j < 3; ++j) ok = ok && map_heads(&p.mapB[j], W[j], dm.H, dm.d, 64, 64);
    if (!ok) return cudaErrorInvalidValue;
    p.src_rows = X;
    p.out[0] = sv.Q;
    p.out[1] = sv.K;
    p.out[2] = sv.V;
    p.T = dm.T;
    p.half = attn_f16(dm) ? 1 : 0;
    if (p.half && dm.rope) {
        p.rope = 1;
        p.rope_tab = make_rope_table(dm.hp, dm.T);
    }
    dim3 grid((p.M + kBM - 1) / kBM, 1, dm.H);
    return launch_kind<kQKV>(p, grid, s);
}

cudaError_t tc_out(const Dims &dm, const void *Wo, const Saved &sv, float *Y, cudaStream_t s,
                   bool zero_output, bool pos_ready) {
    if (use_headsum_out(dm)) {
        if (!pos_ready) {
            cudaError_t e = tc_token_rows(dm, sv, s);
            if (e != cudaSuccess) return e;
        }
        return tc_out_headsum(dm, Wo, sv, Y, s);
    }
    if (zero_output) {
        cudaError_t e = cudaMemsetAsync(Y, 0, sizeof(float) * (size_t)dm.B * dm.T * dm.d, s);
        if (e != cudaSuccess) return e;
    }
    return tc_out_scatter(dm, Wo, sv, Y, s);
}

cudaError_t tc_out_bwd_g(const Dims &dm, const void *Wo, const void *dY, const Saved &sv,
                         cudaStream_t s) {
    // G = dY[I] W_o^T with the row terms fused into the epilogue.
    TcParams p = base_params(dm, sv);
    p.M = p.Mtok;
    p.nkb = (dm.d + kBK - 1) / kBK;
    bool ok = map_gather(&p.mapA, dY, (uint64_t)dm.B * dm.T, dm.d) &&
              map_heads(&p.mapB[0], Wo, dm.H, 64, dm.d, 64);
    if (!ok) return cudaErrorInvalidValue;
    p.src_rows = dY;
    p.ARp = static_cast<const bf16 *>(sv.AR);
    p.out[0] = sv.dA;
    p.out[1] = sv.dQKV;
    p.out_f1 = sv.Dd;
    p.out_f2 = sv.dlogit;
    p.half = attn_f16(dm) ? 1 : 0;
    p.dq16 = dqkv_f16(dm) ? 1 : 0;
    // the k > 128 attention backward (next on this stream) reduce-adds dQ into
    // sv.G: its rows start at zero here, beside dA
    if (dm.k > 128) p.zero_rows = sv.G;
    dim3 grid((p.M + kBM - 1) / kBM, 1, dm.H);
    return launch_kind<kG>(p, grid, s);
}

cudaError_t tc_out_bwd_w(const Dims &dm, const void *dY, const Saved &sv, float *dWo,
                         cudaStream_t s) {
    // dW_o[h](p, c) = sum_m AR(m, p) dY[g(m), c]
    cudaError_t e;
    TcParams q = base_params(dm, sv);
    q.M = dm.d;
    q.nkb = (q.Mtok + kBK - 1) / kBK;
    const int tiles = (dm.d + kBM - 1) / kBM * dm.H;
    q.splits = splits_for(tiles, q.nkb);
    const bool ok = map_gather(&q.mapA, dY, (uint64_t)dm.B * dm.T, dm.d) &&
                    map_heads(&q.mapB[0], sv.AR, dm.H, q.Mtok, 128, 64);
    if (!ok) return cudaErrorInvalidValue;
    q.src_rows = dY;
    q.out_f = dWo;
    if (q.splits > 1) {
        e = cudaMemsetAsync(dWo, 0, sizeof(float) * (size_t)dm.H * 64 * dm.d, s);
        if (e != cudaSuccess) return e;
    }
    dim3 grid2((dm.d + kBM - 1) / kBM, 1, dm.H * q.splits);
    return launch_kind<kDWO>(q, grid2, s);
}

cudaError_t tc_in_bwd(const Dims &dm, const void *Wq, const void *Wk, const void *Wv,
                      const void *Wr, const Saved &sv, float *dX, cudaStream_t s, bool zero_output,
                      bool pos_ready) {
    if (use_headsum_dx(dm)) {
        if (!pos_ready) {
            cudaError_t e = tc_token_rows(dm, sv, s);
            if (e != cudaSuccess) return e;
        }
        return tc_dx_headsum(dm, sv, dX, s);
    }
    if (zero_output) {
        cudaError_t e = cudaMemsetAsync(dX, 0, sizeof(float) * (size_t)dm.B * dm.T * dm.d, s);
        if (e != cudaSuccess) return e;
    }
    (void)Wr;  // read through its fp32 transpose sv.WrT
    return tc_dx(dm, Wq, Wk, Wv, sv, dX, s);
}

cudaError_t tc_w_bwd(const Dims &dm, const void *X, const Saved &sv, float *dWq, float *dWk,
                     float *dWv, float *dWr, cudaStream_t s) {
    TcParams p = base_params(dm, sv);
    p.M = dm.d;
    p.nkb = (p.Mtok + 31) / 32;
    const int tiles = (dm.d + 255) / 256 * dm.H;
    // one wave of single-CTA SMs: the most reduction splits with tiles * splits <= 152
    p.splits = 1;
    while (tiles * p.splits * 2 <= 152 && p.splits * 4 <= p.nkb) p.splits *= 2;
    // fp16 attention path: dQ|dK|dV|dlogit single fp16 rows of 256, and the
    // gathered rows from the fp16 copy of X, one MMA per step
    const bool half = dqkv_f16(dm);
    const void *Xs = half ? sv.X16 : X;
    bool ok = map_gather(&p.mapA, Xs, (uint64_t)dm.B * dm.T, dm.d) &&
              map_heads(&p.mapB[0], sv.dQKV, dm.H, p.Mtok, half ? 256 : kDQKVCols, 32);
    if (!ok) return cudaErrorInvalidValue;
    p.src_rows = Xs;
    p.out_f = dWq;
    p.out_f1 = dWk;
    p.out_f2 = dWv;
    p.out_f3 = dWr;
    if (p.splits > 1) {
        const size_t n = sizeof(float) * (size_t)dm.H * dm.d * 64;
        cudaError_t e;
        if ((e = cudaMemsetAsync(dWq, 0, n, s)) != cudaSuccess) return e;
        if ((e = cudaMemsetAsync(dWk, 0, n, s)) != cudaSuccess) return e;
        if ((e = cudaMemsetAsync(dWv, 0, n, s)) != cudaSuccess) return e;
        if ((e = cudaMemsetAsync(dWr, 0, sizeof(float) * (size_t)dm.d * dm.H, s)) != cudaSuccess)
            return e;
    }
    dim3 grid((dm.d + 255) / 256, 1, dm.H * p.splits);
    return half ? launch_kind<kDWH>(p, grid, s) : launch_kind<kDW>(p, grid, s);
}

}  // namespace mosa
