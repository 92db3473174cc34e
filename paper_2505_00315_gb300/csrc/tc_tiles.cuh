// Shared-memory tile helpers of the attention kernels (tc_attention.cu) and the
// fused per-tile kernels (tc_fused_fwd.cu, tc_fused_bwd.cu): 128-row tiles in
// 64-column blocks of 128-byte-swizzled 16-bit values, stored as bf16 hi / lo
// pairs (v ~ hi + lo) with the split products over them, or as single fp16
// values (k > 128 attention) with one MMA per product.
#pragma once

#include "tc_common.cuh"

namespace mosa {
namespace tc {

constexpr int kTileHalf = 128 * 64 * 2;  // one 64-column block of a 128-row tile, one half: 16 KB

// Tile row r (query or key) of the sequences b0 .. b0+U-1 packed into one tile
// (k rows each): valid when it lies in one of them; lo is the first tile row of
// its sequence (keys c with lo <= c <= r are visible from query r).
struct TileRow {
    bool valid;
    int lo;
};
__device__ __forceinline__ TileRow tile_row(int r, int k, int U, int b0, int B) {
    const int u = r / k;
    return TileRow{u < U && b0 + u < B, u * k};
}

// 32 values v * f as columns c0 .. c0+31 (within one 64-column block) of row r
// of a K-major pair block: hi into hi_blk, lo into lo_blk.
__device__ __forceinline__ void put_pair32(uint8_t *hi_blk, uint8_t *lo_blk, int r, int c0,
                                           const float *v, float f) {
    const int cb = (c0 & 63) >> 3;  // first 16-byte unit within the 128-byte row
#pragma unroll
    for (int c = 0; c < 4; ++c) {
        uint32_t h4[4], l4[4];
#pragma unroll
        for (int e = 0; e < 4; ++e) {
            const float a = v[c * 8 + 2 * e] * f, b = v[c * 8 + 2 * e + 1] * f;
            split_pair2(a, b, h4[e], l4[e]);
        }
        const int off = r * 128 + (((cb + c) ^ (r & 7)) << 4);
        *reinterpret_cast<uint4 *>(hi_blk + off) = make_uint4(h4[0], h4[1], h4[2], h4[3]);
        *reinterpret_cast<uint4 *>(lo_blk + off) = make_uint4(l4[0], l4[1], l4[2], l4[3]);
    }
}

// 32 consecutive keys c0..c0+31 of row r of a [128 x 128] pair tile laid out
// [half][key block].
__device__ __forceinline__ void write_pair32(uint8_t (*tile)[2][kTileHalf], int r, int c0,
                                             const float *v) {
    put_pair32(tile[0][c0 >> 6], tile[1][c0 >> 6], r, c0, v, 1.f);
}

// 32 values v * f as fp16, columns c0 .. c0+31 (within one 64-column block)
// of row r of a K-major fp16 block; returns the largest magnitude written.
__device__ __forceinline__ float put_f16_32(uint8_t *blk, int r, int c0, const float *v, float f) {
    const int cb = (c0 & 63) >> 3;  // first 16-byte unit within the 128-byte row
    float mx = 0.f;
#pragma unroll
    for (int c = 0; c < 4; ++c) {
        uint32_t w[4];
#pragma unroll
        for (int e = 0; e < 4; ++e) {
            const float a = v[c * 8 + 2 * e] * f, b = v[c * 8 + 2 * e + 1] * f;
            mx = fmaxf(mx, fmaxf(fabsf(a), fabsf(b)));
            w[e] = pack_f16x2(a, b);
        }
        const int off = r * 128 + (((cb + c) ^ (r & 7)) << 4);
        *reinterpret_cast<uint4 *>(blk + off) = make_uint4(w[0], w[1], w[2], w[3]);
    }
    return mx;
}

// D (+)= A B over K = 128 for fp16 tiles (one MMA per 16-wide K step), A a
// [128 x 128] tile as two 64-column blocks at a0 and a0 + kTileHalf, B a
// 128-row tile read MN-major (its rows are the K index):
//   a_mn = false: A K-major, K = tile columns (dS K)
//   a_mn = true:  A read as its transpose (P^T dA, dS^T Q), K = tile rows
__device__ __forceinline__ void mma_k128_f16(uint32_t d, uint32_t a0, uint32_t b, bool a_mn,
                                             uint32_t idesc, bool accumulate) {
#pragma unroll
    for (int kk = 0; kk < 8; ++kk) {
        const uint64_t ad = a_mn ? smem_desc_sw128(a0 + kk * 2048, kTileHalf, 1024)
                                 : smem_desc_sw128(a0 + (kk >> 2) * kTileHalf + (kk & 3) * 32, 16, 1024);
        const uint64_t bd = smem_desc_sw128(b + kk * 2048, kTileHalf, 1024);
        mma_bf16(d, ad, bd, idesc, (accumulate || kk > 0) ? 1u : 0u);
    }
}

// D = A B^T over K = 64 for fp16 tiles, both K-major 128-row blocks (S = Q K^T,
// dP = dA V^T; N = 128).
__device__ __forceinline__ void mma_k64_f16(uint32_t d, uint32_t a, uint32_t b, uint32_t idesc) {
#pragma unroll
    for (int kk = 0; kk < 4; ++kk)
        mma_bf16(d, smem_desc_sw128(a + kk * 32, 16, 1024), smem_desc_sw128(b + kk * 32, 16, 1024),
                 idesc, kk > 0 ? 1u : 0u);
}

// Three split products D (+)= Ah Bh + Ah Bl + Al Bh over K = 64.
__device__ __forceinline__ void mma_pair3(uint32_t d, uint32_t a_hi, uint32_t a_lo, uint32_t b_hi,
                                          uint32_t b_lo, bool a_mn, bool b_mn, uint32_t idesc,
                                          bool accumulate_first) {
    const uint32_t aa[3] = {a_hi, a_hi, a_lo}, bb[3] = {b_hi, b_lo, b_hi};
#pragma unroll
    for (int t = 0; t < 3; ++t)
#pragma unroll
        for (int kk = 0; kk < 4; ++kk) {
            const uint64_t ad = a_mn ? smem_desc_sw128(aa[t] + kk * 2048, 8192, 1024)
                                     : smem_desc_sw128(aa[t] + kk * 32, 16, 1024);
            const uint64_t bd = b_mn ? smem_desc_sw128(bb[t] + kk * 2048, 8192, 1024)
                                     : smem_desc_sw128(bb[t] + kk * 32, 16, 1024);
            mma_bf16(d, ad, bd, idesc, (accumulate_first || t > 0 || kk > 0) ? 1u : 0u);
        }
}

// D (+)= A B over K = 128 with A a [128 x 128] pair tile (two 64-wide blocks)
// and B a pair of 128-row tiles, three split products each.
//   a_mn = false: A K-major, K = tile columns (P V, dS K)
//   a_mn = true:  A read as its transpose (P^T dA, dS^T Q), K = tile rows
// With accumulate, the products add to what D already holds.
__device__ __forceinline__ void mma_k128(uint32_t d, const uint8_t (*a)[2][kTileHalf],
                                         const uint8_t (*b)[kTileHalf], bool a_mn, uint32_t idesc,
                                         bool accumulate = false) {
#pragma unroll
    for (int t = 0; t < 3; ++t) {
        const int ah = t == 2 ? 1 : 0, bh = t == 1 ? 1 : 0;
#pragma unroll
        for (int kk = 0; kk < 8; ++kk) {
            uint64_t ad, bd;
            if (a_mn) {
                // rows kk*16.. of both key blocks; next 64-wide M block 16 KB on
                ad = smem_desc_sw128(smem_u32(a[ah][0]) + kk * 2048, kTileHalf, 1024);
            } else {
                ad = smem_desc_sw128(smem_u32(a[ah][kk >> 2]) + (kk & 3) * 32, 16, 1024);
            }
            // B rows = K index (MN-major B: 64-wide N block, 16 rows per step)
            bd = smem_desc_sw128(smem_u32(b[bh]) + kk * 2048, kTileHalf, 1024);
            mma_bf16(d, ad, bd, idesc, (accumulate || t > 0 || kk > 0) ? 1u : 0u);
        }
    }
}

}  // namespace tc
}  // namespace mosa
