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

// One thread per (row, pair): rows of a [rows, 2 * cols] pair array or a
// [rows, cols] fp32 array (Inter<TS>), columns col0 + 2p and col0 + 2p + 1.
template <class TS>
__global__ void rope_rows_kernel(void *p, int cols, int col0, long long rows,
                                 const int32_t *__restrict__ gidx, RopeTable tab, float dir) {
    asm volatile("griddepcontrol.wait;" ::: "memory");
    const long long i = (long long)blockIdx.x * blockDim.x + threadIdx.x;
    if (i >= rows * tab.npairs) return;
    const long long row = i / tab.npairs;
    const int pr = (int)(i - row * tab.npairs);
    const int t = gidx[row] % tab.T;   // gidx = b*T + t
    float x0 = Inter<TS>::ld(p, (size_t)row, cols, col0 + 2 * pr);
    float x1 = Inter<TS>::ld(p, (size_t)row, cols, col0 + 2 * pr + 1);
    rope_turn(x0, x1, tab.phi[pr], t, dir);
    Inter<TS>::st(p, (size_t)row, cols, col0 + 2 * pr, x0);
    Inter<TS>::st(p, (size_t)row, cols, col0 + 2 * pr + 1, x1);
}

}  // namespace

cudaError_t launch_rope(void *p, bool pair, int cols, int col0, long long rows,
                        const int32_t *gidx, const RopeTable &tab, float dir, cudaStream_t s) {
    const long long n = rows * tab.npairs;
    if (n <= 0) return cudaSuccess;
    const dim3 grid((unsigned)((n + 255) / 256));
    cudaError_t e = pair ? launch_pdl(rope_rows_kernel<SplitBF16>, grid, dim3(256), 0, s, p, cols,
                                      col0, rows, gidx, tab, dir)
                         : launch_pdl(rope_rows_kernel<float>, grid, dim3(256), 0, s, p, cols,
                                      col0, rows, gidx, tab, dir);
    note_launches(1);
    return e;
}

}  // namespace mosa
