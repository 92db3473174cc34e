// Host-side launchers of the libmosa kernels (internal; the public C ABI is
// include/mosa.h).  Every launcher enqueues its kernels on `stream` and
// returns the launch status; none synchronizes.
#pragma once

#include <cstdlib>
#include <mutex>
#include <set>
#include <utility>

#include "common.cuh"

namespace mosa {

// Launches `kernel` with programmatic stream serialization when `early` (it
// may begin while the preceding kernel on the stream finishes; the kernel
// itself waits with griddepcontrol.wait before reading that kernel's results).
// A kernel that shares the GPU with another stream's kernel is launched late
// instead: waiting early, its CTAs would hold SMs the other kernel needs.
// MOSA_PDL=0 launches every kernel plainly.
template <class... KArgs, class... Args>
inline cudaError_t launch_ex(bool early, void (*kernel)(KArgs...), dim3 grid, dim3 block,
                             size_t smem, cudaStream_t s, Args &&...args) {
    const char *v = std::getenv("MOSA_PDL");
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = grid;
    cfg.blockDim = block;
    cfg.dynamicSmemBytes = smem;
    cfg.stream = s;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = (!early || (v != nullptr && v[0] == '0')) ? 0 : 1;
    return cudaLaunchKernelEx(&cfg, kernel, std::forward<Args>(args)...);
}
template <typename... KArgs, typename... Args>
inline cudaError_t launch_pdl(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem,
                              cudaStream_t s, Args &&...args) {
    return launch_ex(true, kernel, grid, block, smem, s, std::forward<Args>(args)...);
}

// Raises `kernel`'s dynamic shared-memory limit to `bytes` on the current
// device.  The attribute is per device, so it is set once for each device
// (and each kernel) a process uses; `bytes` must therefore be the largest
// size the kernel is ever launched with, not the size of one launch.
inline cudaError_t allow_smem(const void *kernel, int bytes) {
    static std::mutex mu;
    static std::set<std::pair<int, const void *>> done;
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    std::lock_guard<std::mutex> lk(mu);
    if (done.count({dev, kernel})) return cudaSuccess;
    e = cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, bytes);
    if (e == cudaSuccess) done.insert({dev, kernel});
    return e;
}

// RoPE (Sec. 2.2) angle table for head size hp and sequences of T tokens.
RopeTable make_rope_table(int hp, int T);
// Turns pairs (col0 + 2p, col0 + 2p + 1), p < h'/4, of each of `rows` stored
// rows ([rows, 2 cols] bf16 pairs if `pair`, else [rows, cols] fp32) in place
// by dir * t * theta_p, t = gidx[row] mod T, for two column blocks at once:
// (p0, col0_0) and (p1, col0_1).  col0_* and cols are multiples of 8.
cudaError_t launch_rope(void *p0, int col0_0, void *p1, int col0_1, bool pair, int cols,
                        long long rows, const int32_t *gidx, const RopeTable &tab, float dir,
                        cudaStream_t s);

// F1, Sec. 2.2 router: r_full[b,h,t] = sigmoid(X[b,t,:] . W_r[:,h]) in fp32.
cudaError_t launch_router(const Dims &dm, const void *X, const void *Wr, float *r_full,
                          cudaStream_t stream);
// F1 choosing the tensor-core kernel where it applies.  wr_pad (optional):
// room for a [d, H rounded up to 64] bf16 copy of W_r, used by the
// tensor-core router when H % 64 != 0; zero_status: zero the status word
// first (ordered after all earlier work on the stream).
cudaError_t launch_router_auto(const Dims &dm, const void *X, const void *Wr, float *r_full,
                               uint32_t *status, cudaStream_t stream, void *wr_pad = nullptr,
                               bool zero_status = false);

// F2, Sec. 2.2 TopK: per row of T scores, the k largest (ties: lower index),
// ascending.  If gidx != nullptr, row = b*H + h also writes the head-major
// gather rows gidx[(h*B+b)*k + i] = b*T + I and rsel_hm likewise.
// With first_token, token 0 of every row is kept and the other k-1 are the
// largest of tokens 1..T-1 (Sec. 3.2).
cudaError_t launch_select(int rows, int T, int k, const float *scores, int32_t *I, float *rsel,
                          int B, int H, int32_t *gidx, float *rsel_hm, cudaStream_t stream,
                          bool first_token = false);

// Caller-supplied I / r_sel -> head-major gather rows, validating each row
// (in range, strictly ascending); invalid rows become 0..k-1 and set
// kStatusBadIndex.
cudaError_t launch_indices_to_rows(const Dims &dm, const int32_t *I, const float *rsel,
                                   int32_t *gidx, float *rsel_hm, uint32_t *status,
                                   cudaStream_t stream);

// Dense heads: gidx[(h*B+b)*k + i] = b*T + i (k = T) and rsel_hm = 1.
cudaError_t launch_dense_rows(const Dims &dm, int32_t *gidx, float *rsel_hm,
                              cudaStream_t stream);

// F3: Q, K, V = X[I] W_{q,k,v}[h].
cudaError_t launch_qkv(const Dims &dm, const void *X, const void *Wq, const void *Wk,
                       const void *Wv, const Saved &sv, cudaStream_t stream);

// F4: A = softmax((QK^T + M)/sqrt(h')) V, AR = diag(r) A, lse.
cudaError_t launch_attn_fwd(const Dims &dm, const Saved &sv, cudaStream_t stream);

// F5: Y = 0; Y[b, I, :] += AR W_o[h] summed over heads.
cudaError_t launch_out(const Dims &dm, const void *Wo, const Saved &sv, float *Y,
                       cudaStream_t stream);

// B1: G = dY[I] W_o^T, dr, dA = r G, dlogit, D; dW_o = AR^T dY[I].
cudaError_t launch_out_bwd(const Dims &dm, const void *Wo, const void *dY, const Saved &sv,
                           float *dWo, cudaStream_t stream);

// B2: dQ, dK, dV from dA (flash-style recomputation of P).
cudaError_t launch_attn_bwd(const Dims &dm, const Saved &sv, cudaStream_t stream,
                            float *zero_out = nullptr);

// B3: dX = 0; dX[b, I, :] += dQ W_q^T + dK W_k^T + dV W_v^T + dlogit W_r[:,h]^T.
cudaError_t launch_in_bwd(const Dims &dm, const void *Wq, const void *Wk, const void *Wv,
                          const void *Wr, const Saved &sv, float *dX, cudaStream_t stream);

// B4: dW_{q,k,v}[h] = X[I]^T d{Q,K,V};  dW_r[:,h] = X[I]^T dlogit.
cudaError_t launch_w_bwd(const Dims &dm, const void *X, const Saved &sv, float *dWq,
                         float *dWk, float *dWv, float *dWr, cudaStream_t stream);

// ---- tensor-core path (tc_gemm.cu): bf16 inputs, head size 64 ----
bool tc_supported(const Dims &dm);
// True when the tensor-core kernels serve this shape (false also when the
// environment variable MOSA_FORCE_SIMT is set to a non-zero value).
bool use_tc(const Dims &dm);
// True when the attention runs on fp16 operands (tensor cores, k > 128): Q,
// K, V and dA are then stored as fp16 rows [H, B*k, 64], with RoPE applied
// in the projection's epilogue; otherwise they are bf16 pairs (or fp32).
bool attn_f16(const Dims &dm);
// dQ|dK|dV|dlogit rows as single fp16 ([H, B*k, 256]) for the input- and
// weight-gradient products (with the fp16 copies of X and W_q|W_k|W_v): the
// tensor-core path for k > 128, and for k <= 128 where the weights' copy is
// small (not with the opt-in fused k <= 128 backward, which keeps bf16 pairs).
bool dqkv_f16(const Dims &dm);
// Fused F3 + F4 + F5 for k <= 128 (tc_fused_fwd.cu); off with MOSA_FUSED_FWD=0.
bool tc_fused_forward_supported(const Dims &dm);
bool use_fused_forward(const Dims &dm);
cudaError_t tc_fused_forward(const Dims &dm, const void *X, const void *Wq, const void *Wk,
                             const void *Wv, const void *Wo, const Saved &sv, float *Y,
                             cudaStream_t s);
// Fused G / row terms + attention backward for k <= 128 (tc_fused_bwd.cu);
// opt-in with MOSA_FUSED_BWD=1.
bool use_fused_backward(const Dims &dm);
cudaError_t tc_fused_backward(const Dims &dm, const void *W_o, const void *dY, const Saved &sv,
                              cudaStream_t s);
cudaError_t tc_qkv(const Dims &dm, const void *X, const void *Wq, const void *Wk, const void *Wv,
                   const Saved &sv, cudaStream_t s);
// zero_output = false: the caller has already zeroed Y / dX on this stream's timeline
// (not needed on the token-major path, which writes every element).  pos_ready:
// the token-major path's row map sv.pos has been built on this stream's timeline.
cudaError_t tc_out(const Dims &dm, const void *Wo, const Saved &sv, float *Y, cudaStream_t s,
                   bool zero_output, bool pos_ready = false);
// Token-major products (tc_headsum.cu): every head's rows of a 128-token tile
// summed in TMEM and written once, for layers whose heads keep a large share
// of the tokens: F5 when T <= 2k; B3 (fp16 attention path, H <= 16) only with
// MOSA_HEADSUM=1, which also lifts the T/k limit.  MOSA_HEADSUM=0 turns both off.
bool use_headsum_out(const Dims &dm);
bool use_headsum_dx(const Dims &dm);
// sv.pos[h, b*T + t] = the row b*k + i of head h that holds token t, or -1.
cudaError_t tc_token_rows(const Dims &dm, const Saved &sv, cudaStream_t s);
cudaError_t tc_out_headsum(const Dims &dm, const void *Wo, const Saved &sv, float *Y, cudaStream_t s);
cudaError_t tc_dx_headsum(const Dims &dm, const Saved &sv, float *dX, cudaStream_t s);
// B1 in two independent parts: G and the row terms; dW_o.
cudaError_t tc_out_bwd_g(const Dims &dm, const void *Wo, const void *dY, const Saved &sv,
                         cudaStream_t s);
cudaError_t tc_out_bwd_w(const Dims &dm, const void *dY, const Saved &sv, float *dWo,
                         cudaStream_t s);
cudaError_t tc_in_bwd(const Dims &dm, const void *Wq, const void *Wk, const void *Wv,
                      const void *Wr, const Saved &sv, float *dX, cudaStream_t s,
                      bool zero_output, bool pos_ready = false);
// F5 as a persistent scatter product over (head, 128-row tile, 256-column
// chunk) units: Y[g(m), :] += AR(m, :) W_o[h] (Y zeroed by the caller).
cudaError_t tc_out_scatter(const Dims &dm, const void *Wo, const Saved &sv, float *Y,
                           cudaStream_t s);
// B3 as the same persistent scatter product; needs dX zeroed and sv.WrT
// (tc_transpose_wr).
cudaError_t tc_dx(const Dims &dm, const void *Wq, const void *Wk, const void *Wv, const Saved &sv,
                  float *dX, cudaStream_t s);
// F1 on tensor cores (bf16 inputs, H % 8 == 0); false if not applicable.
// Wr is [d, wr_cols] bf16 with wr_cols >= H (columns beyond H unused).
bool tc_router_applies(const Dims &dm);
bool tc_router(const Dims &dm, const void *X, const void *Wr, int wr_cols, float *r_full,
               uint32_t *status, cudaStream_t s, cudaError_t *err);
// bf16 -> fp16 copy of n values (n % 8 == 0, 16-byte aligned); values beyond
// the fp16 range set kStatusRange.
cudaError_t tc_to_f16(const void *src, void *dst, size_t n, uint32_t *status, cudaStream_t s);
// Address of the fp16 copy of W_o inside sv.W16.
void *wo16_of(const Dims &dm, const Saved &sv);
// fp16 attention path: X -> sv.X16 and W_q, W_k, W_v, W_o -> sv.W16 (bf16 ->
// fp16; out-of-range values set kStatusRange); a null source is skipped.
cudaError_t tc_f16_copies(const Dims &dm, const void *X, const void *Wq, const void *Wk,
                          const void *Wv, const void *Wo, const Saved &sv, cudaStream_t s);
// W_r [d,H] bf16 -> sv.WrT [H,d] fp32 (read by the dX epilogue).
cudaError_t tc_transpose_wr(const Dims &dm, const void *Wr, const Saved &sv, cudaStream_t s);
cudaError_t tc_attn_fwd(const Dims &dm, const Saved &sv, cudaStream_t s);
// For k > 128 the attention backward reduce-adds dQ into the fp32
// accumulator sv.G, whose rows the G kernel (tc_out_bwd_g) zeroes first.
// zero_out (k > 128 only, 16-byte aligned; else nullptr): the layer's dX
// [B*T, d] fp32, zeroed by the kernel beside the attention (see
// attn_bwd_zeroes_dx).
cudaError_t tc_attn_bwd(const Dims &dm, const Saved &sv, cudaStream_t s, float *zero_out = nullptr);
// True when tc_attn_bwd can take over zeroing dX (the fp16 path, k > 128).
inline bool attn_bwd_zeroes_dx(const Dims &dm, const void *dX) {
    return attn_f16(dm) && dX != nullptr && ((uintptr_t)dX % 16) == 0;
}
cudaError_t tc_w_bwd(const Dims &dm, const void *X, const Saved &sv, float *dWq, float *dWk,
                     float *dWv, float *dWr, cudaStream_t s);

}  // namespace mosa
