// Router (F1) and TopK selection (F2) of the MoSA layer, Sec. 2.2:
//   r = sigmoid(X W^r);   r^topk, I = TopK(r, k).
//
// The selection is a per-row radix select on an order-preserving uint32
// image of the fp32 scores (4 passes of 8 bits, most significant first),
// which finds the exact k-th largest key.  With first_token, token 0 gets a
// key above every score's (0xFFFFFFFF; a finite or infinite score maps at most
// to 0xFF800000), so it is always kept and the other k-1 come from the rest.
// A final in-order compaction keeps every key above the k-th largest plus the
// lowest-index keys equal to it, so I comes out
// ascending (the order the causal mask works in) and ties go to the lower
// token index.  Output positions come from one block-wide prefix sum of the
// per-segment counts, so no sort is needed.
#include <algorithm>
#include <mutex>

#include "launch.h"
#include "profile.h"
#include "simt_gemm.cuh"

namespace mosa {
namespace {

template <class E>
struct RouterOp {
    static constexpr bool kAKFast = true;   // X rows are contiguous along d
    static constexpr bool kBKFast = false;  // W_r rows are contiguous along H
    int M, N, K;                            // B*T tokens, H heads, d
    int T, H;
    const E *X, *Wr;
    float *r_full;
    __device__ float a(int, int m, int kk) const { return to_f32(X[(size_t)m * K + kk]); }
    __device__ float b(int, int kk, int n) const { return to_f32(Wr[(size_t)kk * N + n]); }
    __device__ void store(int, int m, int n, float logit) const {
        const int bb = m / T, t = m % T;
        r_full[((size_t)bb * H + n) * T + t] = 1.f / (1.f + expf(-logit));
    }
};

// Order-preserving map of a non-NaN float to uint32 (-0 and +0 map together).
__device__ __forceinline__ uint32_t order_key(float f) {
    uint32_t u = __float_as_uint(f);
    if (u == 0x80000000u) u = 0u;
    return (u & 0x80000000u) ? ~u : (u | 0x80000000u);
}
// The score an order key came from (exact, except that both zeros give +0).
__device__ __forceinline__ float key_score(uint32_t key) {
    return __uint_as_float((key & 0x80000000u) ? (key ^ 0x80000000u) : ~key);
}

constexpr int kSelThreads = 1024;   // upper bound; launches use 256 or 1024
// Rows up to this many scores keep their order keys in shared memory for all
// five passes over them (four radix passes and the compaction).
constexpr int kSelStagedMax = 16384;

// Block-wide exclusive prefix sum of v (thread order); `total` receives the
// sum.  sh has 33 entries.  Two barriers.
__device__ __forceinline__ unsigned long long block_excl_scan(unsigned long long v,
                                                              unsigned long long *sh,
                                                              unsigned long long &total) {
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int nwarps = blockDim.x >> 5;
    unsigned long long incl = v;
#pragma unroll
    for (int off = 1; off < 32; off <<= 1) {
        const unsigned long long y = __shfl_up_sync(0xffffffffu, incl, off);
        if (lane >= off) incl += y;
    }
    if (lane == 31) sh[warp] = incl;
    __syncthreads();
    if (warp == 0) {
        const unsigned long long w = lane < nwarps ? sh[lane] : 0ull;
        unsigned long long wi = w;
#pragma unroll
        for (int off = 1; off < 32; off <<= 1) {
            const unsigned long long y = __shfl_up_sync(0xffffffffu, wi, off);
            if (lane >= off) wi += y;
        }
        sh[lane] = wi - w;
        if (lane == 31) sh[32] = wi;
    }
    __syncthreads();
    total = sh[32];
    return sh[warp] + incl - v;
}

// One CTA per row, 256 to 1024 threads (chosen at launch).
// Radix passes use two histograms in turn (the next one is cleared while the
// current one fills), so a pass costs two barriers; the compaction gives each
// thread a contiguous segment of the row and places its selected keys after
// one block-wide scan of the per-segment counts.
__global__ void __launch_bounds__(kSelThreads)
topk_select_kernel(const float *__restrict__ scores, int T, int k, int32_t *__restrict__ I,
                   float *__restrict__ rsel, int B, int H, int32_t *__restrict__ gidx,
                   float *__restrict__ rsel_hm, int first_token, unsigned long long *span) {
    extern __shared__ uint32_t keys_s[];   // the row's order keys when T <= kSelStagedMax
    __shared__ uint32_t hist[2][256];
    __shared__ unsigned long long sh[33];
    __shared__ uint32_t sh_prefix, sh_remaining, sh_done;
    asm volatile("griddepcontrol.wait;" ::: "memory");  // scores from the router kernel
    span_begin(span);
    const int row = blockIdx.x;
    const float *s = scores + (size_t)row * T;
    const int tid = threadIdx.x;
    const bool staged = T <= kSelStagedMax;
    for (int i = tid; i < 256; i += blockDim.x) hist[0][i] = 0u;
    // token 0's key under first_token: above every score's
    auto key_of = [&](int t) -> uint32_t {
        return (first_token && t == 0) ? 0xFFFFFFFFu : order_key(__ldg(s + t));
    };
    if (staged) {
        if ((T & 3) == 0 && (reinterpret_cast<uintptr_t>(s) & 15u) == 0) {
            // four scores per 16-byte load, the loads of a thread issued together
            const float4 *s4 = reinterpret_cast<const float4 *>(s);
#pragma unroll 4
            for (int q = tid; q < T / 4; q += blockDim.x) {
                const float4 v = __ldg(s4 + q);
                uint4 kk = make_uint4(order_key(v.x), order_key(v.y), order_key(v.z), order_key(v.w));
                if (first_token && q == 0) kk.x = 0xFFFFFFFFu;
                reinterpret_cast<uint4 *>(keys_s)[q] = kk;
            }
        } else {
            for (int t = tid; t < T; t += blockDim.x) keys_s[t] = key_of(t);
        }
    }
    __syncthreads();
    auto key_at = [&](int t) -> uint32_t { return staged ? keys_s[t] : key_of(t); };

    uint32_t prefix = 0u, mask = 0u, remaining = (uint32_t)k;
    for (int pass = 0; pass < 4; ++pass) {
        const int shift = 24 - 8 * pass;
        uint32_t *hc = hist[pass & 1], *hn = hist[(pass + 1) & 1];
        for (int i = tid; i < 256; i += blockDim.x) hn[i] = 0u;  // read by no one this pass
        // (plain shared atomics: measured at 1024 threads and 4096 keys, about
        // 700-800 cycles a pass whether the keys fall into three bins or 256;
        // aggregating equal bins per warp first (match.any) cost 1300-8100)
        for (int t = tid; t < T; t += blockDim.x) {
            const uint32_t key = key_at(t);
            if ((key & mask) == prefix) atomicAdd(&hc[(key >> shift) & 255u], 1u);
        }
        __syncthreads();
        if (tid < 32) {
            // Lane l owns the 8 bins 255-8l ... 248-8l (largest keys first).
            const int lane = tid;
            uint32_t c[8], sum = 0u;
#pragma unroll
            for (int j = 0; j < 8; ++j) {
                c[j] = hc[255 - (lane * 8 + j)];
                sum += c[j];
            }
            uint32_t incl = sum;
#pragma unroll
            for (int off = 1; off < 32; off <<= 1) {
                const uint32_t y = __shfl_up_sync(0xffffffffu, incl, off);
                if (lane >= off) incl += y;
            }
            const uint32_t reach = __ballot_sync(0xffffffffu, incl >= remaining);
            const int first = __ffs(reach) - 1;  // the candidates always number >= remaining
            if (lane == first) {
                uint32_t cum = incl - sum;
                int bin = 0;
                uint32_t left = remaining;
                uint32_t in_bin = 0u;
#pragma unroll
                for (int j = 0; j < 8; ++j) {
                    if (cum + c[j] >= remaining) {
                        bin = 255 - (lane * 8 + j);
                        left = remaining - cum;
                        in_bin = c[j];
                        break;
                    }
                    cum += c[j];
                }
                sh_prefix = prefix | ((uint32_t)bin << shift);
                sh_remaining = left;
                // every key left in the bin is kept: the set is decided
                sh_done = in_bin == left ? 1u : 0u;
            }
        }
        __syncthreads();
        prefix = sh_prefix;
        remaining = sh_remaining;
        mask |= 255u << shift;
        if (sh_done) break;
    }
    // Under `mask` (the bytes decided so far) prefix is now the k-th largest
    // key; the first `remaining` keys equal to it there (in token order) are
    // kept, with every key above it.  When the passes stop early, every key
    // equal to it is kept (`remaining` of them), as the full passes would.
    const uint32_t thr = prefix;
    const int per = (T + (int)blockDim.x - 1) / (int)blockDim.x;
    const int t0 = min(T, tid * per), t1 = min(T, t0 + per);
    uint32_t n_gt = 0u, n_eq = 0u;
    for (int t = t0; t < t1; ++t) {
        const uint32_t key = key_at(t) & mask;
        n_gt += key > thr ? 1u : 0u;
        n_eq += key == thr ? 1u : 0u;
    }
    unsigned long long tot;
    const unsigned long long before =
        block_excl_scan(((unsigned long long)n_gt << 32) | n_eq, sh, tot);
    uint32_t eq_before = (uint32_t)(before & 0xffffffffu);
    uint32_t pos = (uint32_t)(before >> 32) + min(eq_before, remaining);
    const int hh = row % H, bb = row / H;
    for (int t = t0; t < t1 && pos < (uint32_t)k; ++t) {
        const uint32_t full = key_at(t), key = full & mask;
        bool take = key > thr;
        if (key == thr) take = eq_before++ < remaining;
        if (take) {
            // the score from its staged key (no second read of the row), but
            // from memory for token 0 under first_token and for a zero (-0 and
            // +0 share a key)
            const float v = (staged && !(first_token && t == 0) && full != 0x80000000u)
                                ? key_score(full) : __ldg(s + t);
            I[(size_t)row * k + pos] = t;
            rsel[(size_t)row * k + pos] = v;
            if (gidx != nullptr) {
                const size_t o = ((size_t)hh * B + bb) * k + pos;
                gidx[o] = bb * T + t;
                rsel_hm[o] = v;
            }
            ++pos;
        }
    }
    // The next kernel launches only now: launched at this kernel's start, its
    // CTAs (one per SM for the projections) sat on every SM this grid of B*H
    // CTAs leaves idle, and the side stream's copies and zeroing found no SM
    // until the attention kernel's tail (measured at B4 T4096 d1024 H16 k1024:
    // a 13 us wait before the output product, 394 -> 381 us a step).
    asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
    if (span != nullptr) {
        __syncthreads();
        span_end(span);
    }
}

__global__ void indices_to_rows_kernel(const int32_t *__restrict__ I,
                                       const float *__restrict__ rsel, int B, int H, int T,
                                       int k, int32_t *__restrict__ gidx,
                                       float *__restrict__ rsel_hm, uint32_t *status) {
    asm volatile("griddepcontrol.wait;" ::: "memory");
    const int row = blockIdx.x;  // b*H + h
    const int hh = row % H, bb = row / H;
    const int32_t *Ir = I + (size_t)row * k;
    int bad = 0;
    for (int i = threadIdx.x; i < k; i += blockDim.x) {
        const int32_t t = Ir[i];
        if (t < 0 || t >= T || (i > 0 && Ir[i - 1] >= t)) bad = 1;
    }
    bad = __syncthreads_or(bad);
    if (bad && threadIdx.x == 0) atomicOr(status, kStatusBadIndex);
    for (int i = threadIdx.x; i < k; i += blockDim.x) {
        const int32_t t = bad ? i : Ir[i];
        const size_t o = ((size_t)hh * B + bb) * k + i;
        gidx[o] = bb * T + t;
        rsel_hm[o] = rsel[(size_t)row * k + i];
    }
}

// Dense heads (Sec. 2.1, Eq. mha; the dense heads of a hybrid layer,
// Sec. 2.2): every (b, h) keeps all of its k = T tokens with score 1, so row
// m = b*k + i of a head gathers X row b*T + i = m.
__global__ void dense_rows_kernel(long long n, long long rows_per_head,
                                  int32_t *__restrict__ gidx, float *__restrict__ rsel_hm) {
    for (long long o = (long long)blockIdx.x * blockDim.x + threadIdx.x; o < n;
         o += (long long)gridDim.x * blockDim.x) {
        gidx[o] = (int32_t)(o % rows_per_head);
        rsel_hm[o] = 1.f;
    }
}

}  // namespace

cudaError_t launch_router(const Dims &dm, const void *X, const void *Wr, float *r_full,
                          cudaStream_t stream) {
    if (dm.bf16) {
        RouterOp<bf16> op{dm.B * dm.T, dm.H, dm.d, dm.T, dm.H, (const bf16 *)X,
                          (const bf16 *)Wr, r_full};
        return launch_simt_gemm(op, 1, stream);
    }
    RouterOp<float> op{dm.B * dm.T, dm.H, dm.d, dm.T, dm.H, (const float *)X,
                       (const float *)Wr, r_full};
    return launch_simt_gemm(op, 1, stream);
}

// W_r [d,H] -> Wp [d,Hp], columns H..Hp-1 zero, and the status word zeroed
// (status != nullptr).  Launched without the early-launch attribute, so it
// reads W_r and writes the status word only after all earlier work on the
// stream; it lets the router launch early at once (the router still waits for
// its completion before its first load).
__global__ void pad_wr_kernel(const bf16 *__restrict__ Wr, bf16 *__restrict__ Wp, int d, int H,
                              int Hp, uint32_t *status) {
    asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
    if (status != nullptr && blockIdx.x == 0 && threadIdx.x == 0) *status = 0;
    const size_t n = (size_t)d * Hp;
    for (size_t i = (size_t)blockIdx.x * blockDim.x + threadIdx.x; i < n;
         i += (size_t)gridDim.x * blockDim.x) {
        const int c = (int)(i % Hp);
        Wp[i] = c < H ? Wr[(i / Hp) * H + c] : __float2bfloat16(0.f);
    }
}

cudaError_t launch_router_auto(const Dims &dm, const void *X, const void *Wr, float *r_full,
                               uint32_t *status, cudaStream_t stream, void *wr_pad,
                               bool zero_status) {
    cudaError_t e = cudaSuccess;
    const bool tc = use_tc(dm) && tc_router_applies(dm);
    // The tensor-core router loads W_r in blocks of 64 columns; when H is not
    // a multiple of 64 it reads a zero-padded copy, since blocks reaching past
    // column H (filled by the copy engine) ran its main loop at about 60% of
    // the in-bounds speed (10.8 against 6.3 us at B4 T4096 d1024 H8).
    const bool pad = tc && wr_pad != nullptr && dm.H % 64 != 0;
    const int hp64 = (dm.H + 63) / 64 * 64;
    if (pad) {
        const size_t n = (size_t)dm.d * hp64;
        const int grid = (int)std::min<size_t>((n + 255) / 256, 608);
        pad_wr_kernel<<<grid, 256, 0, stream>>>(static_cast<const bf16 *>(Wr),
                                                 static_cast<bf16 *>(wr_pad), dm.d, dm.H, hp64,
                                                 zero_status ? status : nullptr);
        note_launches(1);
        if ((e = cudaGetLastError()) != cudaSuccess) return e;
    } else if (zero_status) {
        if ((e = cudaMemsetAsync(status, 0, sizeof(uint32_t), stream)) != cudaSuccess) return e;
    }
    if (tc && tc_router(dm, X, pad ? wr_pad : Wr, pad ? hp64 : dm.H, r_full, status, stream, &e))
        return e;
    return launch_router(dm, X, Wr, r_full, stream);
}

cudaError_t launch_select(int rows, int T, int k, const float *scores, int32_t *I, float *rsel,
                          int B, int H, int32_t *gidx, float *rsel_hm, cudaStream_t stream,
                          bool first_token) {
    if (rows <= 0) return cudaSuccess;
    const cudaError_t attr =
        allow_smem((const void *)topk_select_kernel, kSelStagedMax * (int)sizeof(uint32_t));
    if (attr != cudaSuccess) return attr;
    const size_t smem = T <= kSelStagedMax ? sizeof(uint32_t) * (size_t)T : 0;
    // about four keys per thread, 256..1024 threads; at most 512 once rows fill
    // the GPU (measured best at rows x T = 128 x 1024, 1024 x 1024, 32..256 x
    // 4096, 512 and 1024 x 4096, 64 x 8192)
    int threads = T / 4 < 256 ? 256 : (T / 4 > 1024 ? 1024 : (T / 4 + 31) / 32 * 32);
    if (rows >= 512 && threads > 512) threads = 512;
    cudaError_t e = launch_pdl(topk_select_kernel, dim3(rows), dim3(threads), smem, stream,
                               scores, T, k, I, rsel, B, H, gidx, rsel_hm, first_token ? 1 : 0,
                               active_span());
    note_launches(1);
    return e;
}

cudaError_t launch_indices_to_rows(const Dims &dm, const int32_t *I, const float *rsel,
                                   int32_t *gidx, float *rsel_hm, uint32_t *status,
                                   cudaStream_t stream) {
    indices_to_rows_kernel<<<dm.B * dm.H, 256, 0, stream>>>(I, rsel, dm.B, dm.H, dm.T, dm.k,
                                                           gidx, rsel_hm, status);
    note_launches(1);
    return cudaGetLastError();
}

cudaError_t launch_dense_rows(const Dims &dm, int32_t *gidx, float *rsel_hm, cudaStream_t stream) {
    const long long n = dm.rows();
    if (n <= 0) return cudaSuccess;
    const long long blocks = (n + 255) / 256;
    dense_rows_kernel<<<(unsigned)(blocks < 4096 ? blocks : 4096), 256, 0, stream>>>(
        n, (long long)dm.B * dm.k, gidx, rsel_hm);
    note_launches(1);
    return cudaGetLastError();
}

}  // namespace mosa
