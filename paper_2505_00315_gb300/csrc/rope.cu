// Rotary position encoding at the tokens' original positions (Sec. 2.2,
// positional encodings): the queries and keys of a head are rotated after the
// projections by angles of the positions t = I[b,h,i] in the full sequence,
// not of the ranks i in the selected subset; half of the head dimensions turn,
// the other half are left unchanged.  Pair p = (2p, 2p+1) of the first h'/2
// dimensions turns by t * theta_p, theta_p = 10000^(-2p / (h'/2)).  The
// backward turns dQ and dK back by the same angles (the rotation's transpose).
//
// This file holds the host-side angle table and the in-place pass over stored
// rows used everywhere except inside the fused forward, which rotates its
// accumulator before splitting it into pairs.
#include <cmath>
#include <cstring>

#include "launch.h"
#include "profile.h"

namespace mosa {

RopeTable make_rope_table(int hp, int T) {
    RopeTable r;
    memset(&r, 0, sizeof(r));
    const int half = hp / 2;
    r.npairs = half / 2;
    r.T = T;
    // theta_p / (2 pi) in turns per position, as a 64-bit fixed-point fraction
    // (theta_p <= 1 rad, so under 0.16 turns: no integer part)
    const double two_pi = 6.283185307179586476925286766559;
    for (int p = 0; p < r.npairs && p < kRopeMaxPairs; ++p) {
        const double theta = std::pow(10000.0, -2.0 * p / (double)half);
        r.phi[p] = (uint64_t)(theta / two_pi * 18446744073709551616.0);
    }
    return r;
}

namespace {

// Eight consecutive values (four pairs) of one stored row: a 16-byte half of
// each bf16 hi/lo pair row, or 32 bytes of an fp32 row.
template <class TS>
struct Oct;

template <>
struct Oct<float> {
    static __device__ __forceinline__ void ld(const void *p, size_t row, int cols, int c, float v[8]) {
        const float4 *q = reinterpret_cast<const float4 *>(static_cast<const float *>(p) + row * cols + c);
        const float4 a = q[0], b = q[1];
        v[0] = a.x; v[1] = a.y; v[2] = a.z; v[3] = a.w;
        v[4] = b.x; v[5] = b.y; v[6] = b.z; v[7] = b.w;
    }
    static __device__ __forceinline__ void st(void *p, size_t row, int cols, int c, const float v[8]) {
        float4 *q = reinterpret_cast<float4 *>(static_cast<float *>(p) + row * cols + c);
        q[0] = make_float4(v[0], v[1], v[2], v[3]);
        q[1] = make_float4(v[4], v[5], v[6], v[7]);
    }
};

template <>
struct Oct<SplitBF16> {
    // value = hi + lo; stored back as hi = rn(v), lo = rn(v - hi), as Inter<SplitBF16>
    static __device__ __forceinline__ void ld(const void *p, size_t row, int cols, int c, float v[8]) {
        const bf16 *q = static_cast<const bf16 *>(p) + row * 2 * cols;
        const uint4 h = *reinterpret_cast<const uint4 *>(q + c);
        const uint4 l = *reinterpret_cast<const uint4 *>(q + cols + c);
        const __nv_bfloat162 *hh = reinterpret_cast<const __nv_bfloat162 *>(&h);
        const __nv_bfloat162 *ll = reinterpret_cast<const __nv_bfloat162 *>(&l);
        for (int j = 0; j < 4; ++j) {
            v[2 * j] = __low2float(hh[j]) + __low2float(ll[j]);
            v[2 * j + 1] = __high2float(hh[j]) + __high2float(ll[j]);
        }
    }
    static __device__ __forceinline__ void st(void *p, size_t row, int cols, int c, const float v[8]) {
        bf16 *q = static_cast<bf16 *>(p) + row * 2 * cols;
        uint4 h, l;
        __nv_bfloat162 *hh = reinterpret_cast<__nv_bfloat162 *>(&h);
        __nv_bfloat162 *ll = reinterpret_cast<__nv_bfloat162 *>(&l);
        for (int j = 0; j < 4; ++j) {
            const bf16 h0 = __float2bfloat16_rn(v[2 * j]), h1 = __float2bfloat16_rn(v[2 * j + 1]);
            hh[j] = __halves2bfloat162(h0, h1);
            ll[j] = __halves2bfloat162(__float2bfloat16_rn(v[2 * j] - __bfloat162float(h0)),
                                       __float2bfloat16_rn(v[2 * j + 1] - __bfloat162float(h1)));
        }
        *reinterpret_cast<uint4 *>(q + c) = h;
        *reinterpret_cast<uint4 *>(q + cols + c) = l;
    }
};

// One thread per (row, segment, group of four pairs): segment s is the
// column block starting at col0[s] of the rows at p[s] (Q and K, or the dQ
// and dK blocks of one dQ|dK|dV row).  groups = h'/16 per segment, a power
// of two (lg = log2).
template <class TS>
__global__ void rope_rows_kernel(void *p0, void *p1, int col0_0, int col0_1, int cols, int lg,
                                 long long rows, const int32_t *__restrict__ gidx, RopeTable tab,
                                 float dir) {
    asm volatile("griddepcontrol.wait;" ::: "memory");
    const long long i = (long long)blockIdx.x * blockDim.x + threadIdx.x;
    const long long row = i >> (lg + 1);
    if (row >= rows) return;
    const int seg = (int)(i >> lg) & 1;
    const int g = (int)i & ((1 << lg) - 1);
    void *p = seg ? p1 : p0;
    const int c = (seg ? col0_1 : col0_0) + 8 * g;
    const int t = gidx[row] % tab.T;   // gidx = b*T + t
    float v[8];
    Oct<TS>::ld(p, (size_t)row, cols, c, v);
    for (int j = 0; j < 4; ++j) rope_turn(v[2 * j], v[2 * j + 1], tab.phi[4 * g + j], t, dir);
    Oct<TS>::st(p, (size_t)row, cols, c, v);
}

}  // namespace

cudaError_t launch_rope(void *p0, int col0_0, void *p1, int col0_1, bool pair, int cols,
                        long long rows, const int32_t *gidx, const RopeTable &tab, float dir,
                        cudaStream_t s) {
    const int groups = tab.npairs / 4;   // h' / 16: 1, 2, 4 or 8
    if (groups < 1 || (groups & (groups - 1)) != 0 || (col0_0 | col0_1 | cols) % 8 != 0)
        return cudaErrorInvalidValue;
    int lg = 0;
    while ((1 << lg) < groups) ++lg;
    const long long n = rows * 2 * groups;
    if (n <= 0) return cudaSuccess;
    const dim3 grid((unsigned)((n + 255) / 256));
    cudaError_t e = pair ? launch_pdl(rope_rows_kernel<SplitBF16>, grid, dim3(256), 0, s, p0, p1,
                                      col0_0, col0_1, cols, lg, rows, gidx, tab, dir)
                         : launch_pdl(rope_rows_kernel<float>, grid, dim3(256), 0, s, p0, p1,
                                      col0_0, col0_1, cols, lg, rows, gidx, tab, dir);
    note_launches(1);
    return e;
}

}  // namespace mosa
