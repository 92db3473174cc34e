// C ABI of libmosa (declared in include/mosa.h): argument validation,
// workspace carving and the launch sequence of the forward and backward
// passes of the MoSA layer (Sec. 2.2, Eq. mosa_mha).
#include <cstdlib>
#include <cstring>
#include <mutex>
#include <unordered_map>

#include "../../include/mosa.h"
#include "launch.h"
#include "profile.h"

namespace mosa {
namespace {

constexpr size_t kAlign = 256;

size_t align_up(size_t x) { return (x + kAlign - 1) / kAlign * kAlign; }

// Validation shared by every entry point: MOSA_OK, INVALID_ARG or UNSUPPORTED.
mosa_status check_shape(const mosa_shape *s, Dims *out) {
    if (s == nullptr) return MOSA_ERR_INVALID_ARG;
    if (s->B <= 0 || s->T <= 0 || s->d <= 0 || s->H <= 0 || s->hp <= 0 || s->k <= 0)
        return MOSA_ERR_INVALID_ARG;
    if (s->k > s->T) return MOSA_ERR_INVALID_ARG;
    if (s->dtype != MOSA_F32 && s->dtype != MOSA_BF16) return MOSA_ERR_INVALID_ARG;
    if (s->first_token != 0 && s->first_token != 1) return MOSA_ERR_INVALID_ARG;
    if (s->rope != 0 && s->rope != 1) return MOSA_ERR_INVALID_ARG;
    const long long lim = 1LL << 31;
    if ((long long)s->B * s->T * s->d >= lim) return MOSA_ERR_UNSUPPORTED;
    if ((long long)s->H * s->d * s->hp >= lim) return MOSA_ERR_UNSUPPORTED;
    if ((long long)s->B * s->H * s->T >= lim) return MOSA_ERR_UNSUPPORTED;
    if ((long long)s->B * s->H * s->k * 3 * s->hp >= lim) return MOSA_ERR_UNSUPPORTED;
    if (s->T > 65536) return MOSA_ERR_UNSUPPORTED;
    if (s->H > 65535) return MOSA_ERR_UNSUPPORTED;
    if (s->d % 8 != 0) return MOSA_ERR_UNSUPPORTED;
    if (s->hp != 16 && s->hp != 32 && s->hp != 64 && s->hp != 128) return MOSA_ERR_UNSUPPORTED;
    if (out)
        *out = Dims{s->B, s->T, s->d, s->H, s->hp, s->k, s->dtype == MOSA_BF16, s->first_token != 0,
                    s->rope != 0};
    return MOSA_OK;
}

// Carves the workspace; returns the bytes needed (and fills *sv if base != nullptr).
size_t carve(const Dims &dm, char *base, Saved *sv) {
    size_t off = 0;
    auto take = [&](size_t bytes) -> char * {
        char *p = base ? base + off : nullptr;
        off += align_up(bytes);
        return p;
    };
    const size_t R = (size_t)dm.rows();
    const size_t e = 4;  // fp32, or a bf16 hi/lo pair
    Saved s{};
    s.status = (uint32_t *)take(sizeof(uint32_t));
    s.r_full = (float *)take(sizeof(float) * (size_t)dm.B * dm.H * dm.T);
    s.gidx = (int32_t *)take(sizeof(int32_t) * R);
    s.rsel = (float *)take(sizeof(float) * R);
    s.Q = take(e * R * dm.hp);
    s.K = take(e * R * dm.hp);
    s.V = take(e * R * dm.hp);
    s.A = (float *)take(sizeof(float) * R * dm.hp);
    s.AR = take(e * R * dm.hp);
    s.lse = (float *)take(sizeof(float) * R);
    s.dA = take(e * R * dm.hp);
    s.dlogit = (float *)take(sizeof(float) * R);
    s.Dd = (float *)take(sizeof(float) * R);
    s.dQKV = take(e * R * 4 * dm.hp);  // 3 h' columns, or 4 blocks of 64 on the tensor cores
    s.G = (float *)take(sizeof(float) * R * dm.hp);
    s.WrT = (float *)take(sizeof(float) * (size_t)dm.d * dm.H);
    // (reserved for either dtype, so that the size depends on the shape only)
    if (dm.H % 64 != 0) s.Wr64 = take((size_t)2 * dm.d * ((dm.H + 63) / 64 * 64));
    s.spans = (unsigned long long *)take(sizeof(unsigned long long) * 2 * 16);
    // the fp16 copies of the tensor-core path (reserved whenever that path can
    // run, so the size does not depend on the environment's kernel-path switches)
    if (dm.bf16 && dm.hp == 64) {
        s.X16 = take((size_t)2 * dm.B * dm.T * dm.d);
        s.W16 = take((size_t)2 * 4 * dm.H * dm.d * dm.hp);   // W_q, W_k, W_v, W_o
    }
    if (dm.bf16 && dm.hp == 64 && dm.k > 128) {
        s.AR16 = take((size_t)2 * R * dm.hp);
        s.pos = (int32_t *)take(sizeof(int32_t) * (size_t)dm.H * dm.B * dm.T);
    }
    if (sv) *sv = s;
    return off;
}

mosa_status check_workspace(const Dims &dm, void *ws, size_t bytes, Saved *sv) {
    if (ws == nullptr || ((uintptr_t)ws % kAlign) != 0) return MOSA_ERR_WORKSPACE;
    if (bytes < carve(dm, nullptr, nullptr)) return MOSA_ERR_WORKSPACE;
    carve(dm, (char *)ws, sv);
    return MOSA_OK;
}

mosa_status cuda_status(cudaError_t e) { return e == cudaSuccess ? MOSA_OK : MOSA_ERR_CUDA; }

// Stages of a forward call and of a backward call (timeline slot resets).
constexpr uint32_t kForwardStages = (1u << kStageRouter) | (1u << kStageSelect) | (1u << kStageQkv) |
                                    (1u << kStageAttnFwd) | (1u << kStageOut) | (1u << kStageFwdUnit);
constexpr uint32_t kBackwardStages = (1u << kStageOutBwd) | (1u << kStageAttnBwd) |
                                     (1u << kStageInBwd) | (1u << kStageWBwd) | (1u << kStageDwo) |
                                     (1u << kStageBwdUnit);

#define MOSA_TRY(expr)                                  \
    do {                                                \
        cudaError_t _e = (expr);                        \
        if (_e != cudaSuccess) return MOSA_ERR_CUDA;    \
    } while (0)

// ------------------------------------------------ concurrent branches
// On the tensor-core path independent kernels run on a second, internal
// stream joined back with events (graph branches when captured):
//   forward:  zeroing Y and (fp16 attention path) the fp16 copies of X and
//             W_q|W_k|W_v run beside TopK (forked after the router, joined
//             before the output product);
//   backward: dW_o, the W_r transpose and (except on the fp16 path, where
//             the attention backward does it) the zeroing of dX run beside
//             G -> attention backward; then dX and dW run side by side.
// A hybrid call runs the MoSA heads and then the dense heads, each this way.
struct DevResources {
    cudaStream_t side = nullptr;
    cudaEvent_t ev[4] = {};
};
constexpr int kMaxDev = 64;
std::mutex g_res_mu;
DevResources g_res[kMaxDev];

DevResources *dev_resources() {
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDev) return nullptr;
    std::lock_guard<std::mutex> lk(g_res_mu);
    DevResources &r = g_res[dev];
    if (r.side == nullptr) {
        if (cudaStreamCreateWithFlags(&r.side, cudaStreamNonBlocking) != cudaSuccess) {
            r.side = nullptr;
            return nullptr;
        }
        for (auto &e : r.ev)
            if (cudaEventCreateWithFlags(&e, cudaEventDisableTiming) != cudaSuccess) return nullptr;
    }
    return &r;
}

// `to` waits for the work enqueued so far on `from`.
cudaError_t link(cudaStream_t from, cudaStream_t to, cudaEvent_t ev) {
    cudaError_t e = cudaEventRecord(ev, from);
    return e != cudaSuccess ? e : cudaStreamWaitEvent(to, ev, 0);
}

// F3-F5 for the rows already selected into sv.gidx / sv.rsel.
// RoPE (Sec. 2.2) in place on the stored Q and K rows (dir +1), or on the dQ
// and dK blocks of the dQ|dK|dV rows (dir -1).  Pair storage for bf16 inputs:
// on the tensor cores Q is [hi 64 | lo 64] and dQ|dK|dV|dlogit [hi 256 | lo 256]
// per row, on the CUDA cores [hi hp | lo hp] and [hi 3hp | lo 3hp]; fp32 rows
// otherwise.
cudaError_t rope_qk(const Dims &dm, const Saved &sv, bool grads, cudaStream_t s) {
    const RopeTable tab = make_rope_table(dm.hp, dm.T);
    const long long rows = dm.rows();
    const bool pair = dm.bf16;
    if (!grads) return launch_rope(sv.Q, 0, sv.K, 0, pair, dm.hp, rows, sv.gidx, tab, 1.f, s);
    const int cols = use_tc(dm) ? 256 : 3 * dm.hp;
    return launch_rope(sv.dQKV, 0, sv.dQKV, dm.hp, pair, cols, rows, sv.gidx, tab, -1.f, s);
}

mosa_status forward_heads(const Dims &dm, const void *X, const void *W_q, const void *W_k,
                          const void *W_v, const void *W_o, float *Y, const Saved &sv,
                          cudaStream_t s) {
    {
        StageScope st_(kStageQkv, s);
        MOSA_TRY(launch_qkv(dm, X, W_q, W_k, W_v, sv, s));
        // (the fp16 attention path turns Q and K in the projection's epilogue)
        if (dm.rope && !attn_f16(dm)) MOSA_TRY(rope_qk(dm, sv, false, s));
    }
    {
        StageScope st_(kStageAttnFwd, s);
        MOSA_TRY(launch_attn_fwd(dm, sv, s));
    }
    {
        StageScope st_(kStageOut, s);
        MOSA_TRY(launch_out(dm, W_o, sv, Y, s));
    }
    return MOSA_OK;
}

// Tensor-core forward: a chain of kernels on the caller's stream, each launched
// early (programmatic dependent launch).  Y is zeroed on the side stream,
// forked after the router and joined before the output product (measured:
// forked before the router, the zeroing slowed the router's single short wave
// at B8 T1024 d512 H16 k128 by about 8 us per step).
mosa_status forward_tc(const Dims &dm, const void *X, const void *W_r, const void *W_q,
                       const void *W_k, const void *W_v, const void *W_o, float *Y, int32_t *I,
                       float *r_sel, float *rf, bool route, const int32_t *I_in,
                       const float *rsel_in, const Saved &sv, cudaStream_t s, DevResources &r) {
    set_span_base(sv.spans);   // measurement: this call's kernel-span slots
    MOSA_TRY(begin_timeline_call(kForwardStages, s));
    const size_t ny = (size_t)dm.B * dm.T * dm.d;
    // A call that adds into Y continues the status word of the call that wrote it.
    if (route) {
        StageScope st_(kStageRouter, s);
        MOSA_TRY(launch_router_auto(dm, X, W_r, rf, sv.status, s, sv.Wr64, !dm.accumulate));
    } else if (!dm.accumulate) {
        MOSA_TRY(cudaMemsetAsync(sv.status, 0, sizeof(uint32_t), s));
    }
    MOSA_TRY(link(s, r.side, r.ev[0]));
    // (the token-major output product writes every element of Y itself)
    const bool headsum = !use_fused_forward(dm) && use_headsum_out(dm);
    if (!dm.accumulate && !headsum) MOSA_TRY(cudaMemsetAsync(Y, 0, sizeof(float) * ny, r.side));
    // the fused k <= 128 kernel needs only Y zeroed from the side stream
    const bool fused = use_fused_forward(dm);
    if (fused) MOSA_TRY(cudaEventRecord(r.ev[1], r.side));
    // the fp16 copies of X and W_q|W_k|W_v that the backward's products with
    // single-fp16 dQ|dK|dV read, and (k > 128) of W_o for the output product,
    // made here beside TopK, whose grid (one CTA per (b, h) row) leaves most
    // SMs idle
    if (dqkv_f16(dm))
        MOSA_TRY(tc_f16_copies(dm, X, W_q, W_k, W_v, attn_f16(dm) ? W_o : nullptr, sv, r.side));
    if (route) {
        StageScope st_(kStageSelect, s);
        MOSA_TRY(launch_select(dm.B * dm.H, dm.T, dm.k, rf, I, r_sel, dm.B, dm.H, sv.gidx,
                               sv.rsel, s, dm.first_token));
    } else if (I_in == nullptr) {
        StageScope st_(kStageSelect, s);
        MOSA_TRY(launch_dense_rows(dm, sv.gidx, sv.rsel, s));
    } else {
        StageScope st_(kStageSelect, s);
        MOSA_TRY(launch_indices_to_rows(dm, I_in, rsel_in, sv.gidx, sv.rsel, sv.status, s));
    }
    if (headsum) {
        // the token-major output product's row map, beside the projection and attention
        MOSA_TRY(link(s, r.side, r.ev[2]));
        MOSA_TRY(tc_token_rows(dm, sv, r.side));
    }
    if (fused) {
        MOSA_TRY(cudaStreamWaitEvent(s, r.ev[1], 0));  // Y zeroed
        {
            StageScope st_(kStageFwdUnit, s);
            MOSA_TRY(tc_fused_forward(dm, X, W_q, W_k, W_v, W_o, sv, Y, s));
        }
        MOSA_TRY(link(r.side, s, r.ev[3]));  // the backward's fp16 copies
        return MOSA_OK;
    }
    {
        StageScope st_(kStageQkv, s);
        MOSA_TRY(launch_qkv(dm, X, W_q, W_k, W_v, sv, s));
        // (the fp16 attention path turns Q and K in the projection's epilogue)
        if (dm.rope && !attn_f16(dm)) MOSA_TRY(rope_qk(dm, sv, false, s));
    }
    {
        StageScope st_(kStageAttnFwd, s);
        MOSA_TRY(launch_attn_fwd(dm, sv, s));
    }
    MOSA_TRY(link(r.side, s, r.ev[1]));  // Y zeroed, or the row map built
    {
        StageScope st_(kStageOut, s);
        MOSA_TRY(tc_out(dm, W_o, sv, Y, s, false, headsum));
    }
    return MOSA_OK;
}

// Tensor-core backward.  Main stream: G and the row terms, the attention
// backward (zeroing dX on the fp16 path), then dX.  Side stream: dW_o beside
// G, the W_r transpose and otherwise the zeroing of dX, then dW once
// dQ|dK|dV|dlogit exist; the main stream waits for the side stream only
// before dX and at the final join.
mosa_status backward_tc(const Dims &dm, const void *X, const void *W_r, const void *W_q,
                        const void *W_k, const void *W_v, const void *W_o, const void *dY,
                        float *dX, float *dW_r, float *dW_q, float *dW_k, float *dW_v,
                        float *dW_o, const Saved &sv, cudaStream_t s, DevResources &r) {
    set_span_base(sv.spans);   // measurement: this call's kernel-span slots
    MOSA_TRY(begin_timeline_call(kBackwardStages, s));   // before the side stream forks
    cudaStream_t t = r.side;
    const size_t nx = (size_t)dm.B * dm.T * dm.d;
    MOSA_TRY(link(s, t, r.ev[0]));
    if (use_fused_backward(dm)) {
        // The fused kernel (G, row terms, attention backward) holds a whole SM
        // per CTA, so nothing runs beside it; dX, dW and dW_o then share the GPU.
        MOSA_TRY(tc_transpose_wr(dm, W_r, sv, t));
        if (!dm.accumulate) MOSA_TRY(cudaMemsetAsync(dX, 0, sizeof(float) * nx, t));
        MOSA_TRY(cudaEventRecord(r.ev[1], t));  // dX zeroed, W_r transposed
        {
            StageScope st_(kStageBwdUnit, s);
            MOSA_TRY(tc_fused_backward(dm, W_o, dY, sv, s));
            if (dm.rope) MOSA_TRY(rope_qk(dm, sv, true, s));
        }
        MOSA_TRY(link(s, t, r.ev[2]));  // dQ|dK|dV|dlogit ready
        {
            StageScope st_(kStageDwo, t);
            MOSA_TRY(tc_out_bwd_w(dm, dY, sv, dW_o, t));
        }
        {
            StageScope st_(kStageWBwd, t);
            MOSA_TRY(tc_w_bwd(dm, X, sv, dW_q, dW_k, dW_v, dW_r, t));
        }
        MOSA_TRY(cudaStreamWaitEvent(s, r.ev[1], 0));
        {
            StageScope st_(kStageInBwd, s);
            MOSA_TRY(tc_in_bwd(dm, W_q, W_k, W_v, W_r, sv, dX, s, false));
        }
        MOSA_TRY(link(t, s, r.ev[3]));  // join
        return MOSA_OK;
    }
    // (the fp16 attention path's copies of X and W_q|W_k|W_v were made by the forward)
    MOSA_TRY(tc_transpose_wr(dm, W_r, sv, t));
    // The token-major dX product writes every element of dX itself, from the
    // token-to-row map sv.pos that the forward built (use_headsum_dx implies
    // use_headsum_out); the token-major G reads that map too, so nothing
    // rewrites it here.
    const bool headsum = use_headsum_dx(dm);
    // dX starts at zero for the scatter-add product: on the fp16 path the
    // attention backward's idle warps zero it (a 67 MB memset on the side
    // stream found no free SM until that kernel's tail and delayed dX)
    const bool zero_in_attn = !headsum && !dm.accumulate && attn_bwd_zeroes_dx(dm, dX);
    if (!headsum && !dm.accumulate && !zero_in_attn)
        MOSA_TRY(cudaMemsetAsync(dX, 0, sizeof(float) * nx, t));
    MOSA_TRY(cudaEventRecord(r.ev[1], t));  // dX zeroed (unless by the attention backward), W_r transposed
    {
        // dW_o after the event dX waits for, so that dX does not wait for it
        StageScope st_(kStageDwo, t);
        MOSA_TRY(tc_out_bwd_w(dm, dY, sv, dW_o, t));
    }
    {
        StageScope st_(kStageOutBwd, s);
        MOSA_TRY(tc_out_bwd_g(dm, W_o, dY, sv, s));
    }
    {
        StageScope st_(kStageAttnBwd, s);
        MOSA_TRY(launch_attn_bwd(dm, sv, s, zero_in_attn ? dX : nullptr));
        // (the fp16 rows have dQ and dK turned back before rounding)
        if (dm.rope && !dqkv_f16(dm)) MOSA_TRY(rope_qk(dm, sv, true, s));
    }
    MOSA_TRY(link(s, t, r.ev[2]));  // dQ|dK|dV|dlogit ready for dW
    {
        StageScope st_(kStageWBwd, t);
        MOSA_TRY(tc_w_bwd(dm, X, sv, dW_q, dW_k, dW_v, dW_r, t));
    }
    MOSA_TRY(cudaStreamWaitEvent(s, r.ev[1], 0));  // W_r transposed (and dX zeroed on the side)
    {
        StageScope st_(kStageInBwd, s);
        MOSA_TRY(tc_in_bwd(dm, W_q, W_k, W_v, W_r, sv, dX, s, false, /*pos_ready=*/true));
    }
    MOSA_TRY(link(t, s, r.ev[3]));  // join
    return MOSA_OK;
}

// The launch sequences of the three calls, on stream s.  `res` is the side
// stream of the tensor-core path (nullptr: the CUDA-core sequence).

// Router, TopK and the heads (mosa_forward).
mosa_status forward_routed(const Dims &dm, const void *X, const void *W_r, const void *W_q,
                           const void *W_k, const void *W_v, const void *W_o, float *Y,
                           int32_t *I, float *r_sel, float *rf, const Saved &sv, cudaStream_t s,
                           DevResources *res) {
    set_span_base(sv.spans);   // measurement: this call's kernel-span slots
    if (res != nullptr)
        return forward_tc(dm, X, W_r, W_q, W_k, W_v, W_o, Y, I, r_sel, rf, true, nullptr, nullptr,
                          sv, s, *res);
    MOSA_TRY(begin_timeline_call(kForwardStages, s));
    MOSA_TRY(cudaMemsetAsync(sv.status, 0, sizeof(uint32_t), s));
    {
        StageScope st_(kStageRouter, s);
        MOSA_TRY(launch_router_auto(dm, X, W_r, rf, sv.status, s));
    }
    {
        StageScope st_(kStageSelect, s);
        MOSA_TRY(launch_select(dm.B * dm.H, dm.T, dm.k, rf, I, r_sel, dm.B, dm.H, sv.gidx,
                               sv.rsel, s, dm.first_token));
    }
    return forward_heads(dm, X, W_q, W_k, W_v, W_o, Y, sv, s);
}

// The heads on given token sets (mosa_forward_with_indices); I == nullptr:
// every token with score 1 (dense heads, k = T).
mosa_status forward_given(const Dims &dm, const void *X, const void *W_q, const void *W_k,
                          const void *W_v, const void *W_o, const int32_t *I,
                          const float *r_sel, float *Y, const Saved &sv, cudaStream_t s,
                          DevResources *res) {
    set_span_base(sv.spans);   // measurement: this call's kernel-span slots
    if (res != nullptr)
        return forward_tc(dm, X, nullptr, W_q, W_k, W_v, W_o, Y, nullptr, nullptr, nullptr, false,
                          I, r_sel, sv, s, *res);
    MOSA_TRY(begin_timeline_call(kForwardStages, s));
    if (!dm.accumulate) MOSA_TRY(cudaMemsetAsync(sv.status, 0, sizeof(uint32_t), s));
    {
        StageScope st_(kStageSelect, s);
        if (I == nullptr)
            MOSA_TRY(launch_dense_rows(dm, sv.gidx, sv.rsel, s));
        else
            MOSA_TRY(launch_indices_to_rows(dm, I, r_sel, sv.gidx, sv.rsel, sv.status, s));
    }
    return forward_heads(dm, X, W_q, W_k, W_v, W_o, Y, sv, s);
}

// The backward (mosa_backward).
mosa_status backward_all(const Dims &dm, const void *X, const void *W_r, const void *W_q,
                         const void *W_k, const void *W_v, const void *W_o, const void *dY,
                         float *dX, float *dW_r, float *dW_q, float *dW_k, float *dW_v,
                         float *dW_o, const Saved &sv, cudaStream_t s, DevResources *res) {
    set_span_base(sv.spans);   // measurement: this call's kernel-span slots
    if (res != nullptr)
        return backward_tc(dm, X, W_r, W_q, W_k, W_v, W_o, dY, dX, dW_r, dW_q, dW_k, dW_v, dW_o,
                           sv, s, *res);
    MOSA_TRY(begin_timeline_call(kBackwardStages, s));
    {
        StageScope st_(kStageOutBwd, s);
        MOSA_TRY(launch_out_bwd(dm, W_o, dY, sv, dW_o, s));
    }
    {
        StageScope st_(kStageAttnBwd, s);
        MOSA_TRY(launch_attn_bwd(dm, sv, s));
        if (dm.rope) MOSA_TRY(rope_qk(dm, sv, true, s));
    }
    {
        StageScope st_(kStageInBwd, s);
        MOSA_TRY(launch_in_bwd(dm, W_q, W_k, W_v, W_r, sv, dX, s));
    }
    {
        StageScope st_(kStageWBwd, s);
        MOSA_TRY(launch_w_bwd(dm, X, sv, dW_q, dW_k, dW_v, dW_r, s));
    }
    return MOSA_OK;
}

// ------------------------------------------------------------ hybrid layers
// MoSA heads plus dense heads (Sec. 2.2, hybridization) or local heads
// (Sec. 3.4).  The dense heads run through the given-token-set path with
// every token and unit scores: with r = 1 the router terms vanish (dlogit =
// D (1 - r) = 0), so they get a zeroed W_r and a scratch dW_r.  Local heads
// (causal attention within blocks of w tokens) are dense heads over B*T/w
// sequences of w tokens, the same rows of X, Y and dX; RoPE scores depend on
// position differences only, so positions counted from each block's start
// give the same attention.  The dense heads add into the Y and dX the MoSA
// heads wrote.
struct Hybrid {
    Dims sparse, dense;
    bool has_dense;
};

mosa_status check_hybrid(const mosa_hybrid_shape *hs, Hybrid *h) {
    if (hs == nullptr) return MOSA_ERR_INVALID_ARG;
    mosa_status st = check_shape(&hs->sparse, &h->sparse);
    if (st != MOSA_OK) return st;
    const int T = hs->sparse.T;
    if (hs->H_dense < 0 || hs->window < 0 || hs->window > T) return MOSA_ERR_INVALID_ARG;
    h->has_dense = hs->H_dense > 0;
    h->dense = Dims{};
    if (!h->has_dense) return MOSA_OK;
    const int w = hs->window == 0 ? T : hs->window;
    if (T % w != 0) return MOSA_ERR_UNSUPPORTED;
    mosa_shape ds = hs->sparse;
    ds.B = hs->sparse.B * (T / w);
    ds.T = w;
    ds.H = hs->H_dense;
    ds.k = w;
    ds.first_token = 0;
    if ((st = check_shape(&ds, &h->dense)) != MOSA_OK) return st;
    h->dense.accumulate = true;
    return MOSA_OK;
}

struct HybridSpace {
    Saved sparse, dense;
    void *zero_wr;    // [d, H_dense] zeros in the storage dtype
    float *dwr;       // [d, H_dense] fp32, discarded
    size_t zero_wr_bytes;
};

// Sparse heads' state, then the dense heads' (sharing the status word), then
// the two W_r stand-ins.  Returns the bytes needed.
size_t carve_hybrid(const Hybrid &h, char *base, HybridSpace *sp) {
    Saved ss{}, ds{};
    const size_t o1 = carve(h.sparse, base, &ss);
    size_t total = o1;
    size_t nwr = 0;
    char *dense_base = base ? base + o1 : nullptr;
    if (h.has_dense) {
        const size_t o2 = carve(h.dense, dense_base, &ds);
        nwr = (size_t)h.dense.d * h.dense.H * h.dense.esize();
        total = o1 + o2 + align_up(nwr) + align_up(sizeof(float) * h.dense.d * h.dense.H);
        if (base) {
            ds.status = ss.status;
            sp->zero_wr = base + o1 + o2;
            sp->dwr = (float *)(base + o1 + o2 + align_up(nwr));
        }
    }
    if (base) {
        sp->sparse = ss;
        sp->dense = ds;
        sp->zero_wr_bytes = nwr;
        if (!h.has_dense) {
            sp->zero_wr = nullptr;
            sp->dwr = nullptr;
        }
    }
    return total;
}

mosa_status check_hybrid_workspace(const Hybrid &h, void *ws, size_t bytes, HybridSpace *sp) {
    if (ws == nullptr || ((uintptr_t)ws % kAlign) != 0) return MOSA_ERR_WORKSPACE;
    if (bytes < carve_hybrid(h, nullptr, nullptr)) return MOSA_ERR_WORKSPACE;
    carve_hybrid(h, (char *)ws, sp);
    return MOSA_OK;
}

// ---------------------------------------------------------- graph cache
// A layer call enqueues about a dozen kernels and memsets; launched one by one
// from the host that costs tens of microseconds per call.  The first call with
// a given shape, set of pointers, kernel path and stage-timing mask is captured
// on an internal stream into a CUDA graph; later identical calls launch that
// graph on the caller's stream.  MOSA_GRAPHS=0 turns this off.

struct GraphKey {
    int op, device, tc;
    uint32_t mask;
    mosa_shape shape;
    int extra[2];  // hybrid calls: dense heads, window
    const void *ptr[28];
    bool operator==(const GraphKey &o) const { return std::memcmp(this, &o, sizeof(GraphKey)) == 0; }
};

struct GraphKeyHash {
    size_t operator()(const GraphKey &k) const {
        const unsigned char *b = reinterpret_cast<const unsigned char *>(&k);
        uint64_t h = 1469598103934665603ull;
        for (size_t i = 0; i < sizeof(GraphKey); ++i) h = (h ^ b[i]) * 1099511628211ull;
        return (size_t)h;
    }
};

struct GraphEntry {
    cudaGraphExec_t exec = nullptr;
    CaptureRecord rec;
};

constexpr size_t kMaxGraphs = 128;
constexpr int kMaxDevices = 64;
std::mutex g_graph_mu;
std::unordered_map<GraphKey, GraphEntry *, GraphKeyHash> g_graphs;
cudaStream_t g_capture_stream[kMaxDevices] = {};

bool graphs_enabled() {
    const char *v = std::getenv("MOSA_GRAPHS");
    return v == nullptr || v[0] != '0';
}

int path_bits(const Dims &dm) {
    return (use_tc(dm) ? 1 : 0) | (use_fused_forward(dm) ? 2 : 0) | (use_fused_backward(dm) ? 4 : 0) |
           (use_headsum_out(dm) ? 8 : 0) | (use_headsum_dx(dm) ? 16 : 0);
}

GraphKey make_key(int op, const Dims &dm, const mosa_shape *shape,
                  std::initializer_list<const void *> ptrs, const Dims *dense = nullptr,
                  int extra0 = 0, int extra1 = 0) {
    GraphKey k;
    std::memset(&k, 0, sizeof(k));
    k.op = op;
    cudaGetDevice(&k.device);
    k.tc = path_bits(dm) | (dense ? path_bits(*dense) << 5 : 0);
    k.mask = profile_mask();
    k.shape = *shape;
    k.extra[0] = extra0;
    k.extra[1] = extra1;
    int i = 0;
    for (const void *p : ptrs) k.ptr[i++] = p;
    return k;
}

// Runs `enqueue(stream)`, through a cached CUDA graph when possible.
template <class Enqueue>
mosa_status run_graphed(const GraphKey &key, cudaStream_t user, Enqueue &&enqueue) {
    // One lock for both paths: the eager path shares the internal side stream
    // and its events between calls.
    std::lock_guard<std::mutex> lk(g_graph_mu);
    if (!graphs_enabled() || key.device < 0 || key.device >= kMaxDevices) return enqueue(user);
    auto it = g_graphs.find(key);
    GraphEntry *e = it == g_graphs.end() ? nullptr : it->second;
    if (e == nullptr) {
        if (g_graphs.size() >= kMaxGraphs) return enqueue(user);
        cudaStream_t &cs = g_capture_stream[key.device];
        if (cs == nullptr && cudaStreamCreateWithFlags(&cs, cudaStreamNonBlocking) != cudaSuccess) {
            cs = nullptr;
            return enqueue(user);
        }
        e = new GraphEntry;
        capture_into(&e->rec);
        mosa_status st = MOSA_ERR_CUDA;
        cudaGraph_t g = nullptr;
        if (cudaStreamBeginCapture(cs, cudaStreamCaptureModeThreadLocal) == cudaSuccess) {
            st = enqueue(cs);
            if (cudaStreamEndCapture(cs, &g) != cudaSuccess) st = MOSA_ERR_CUDA;
        }
        capture_into(nullptr);
        if (st == MOSA_OK && g != nullptr && cudaGraphInstantiate(&e->exec, g, 0) != cudaSuccess)
            st = MOSA_ERR_CUDA;
        if (g != nullptr) cudaGraphDestroy(g);
        if (st != MOSA_OK) {
            (void)cudaGetLastError();
            for (auto &q : e->rec.pairs) {
                cudaEventDestroy(q.start);
                cudaEventDestroy(q.stop);
            }
            delete e;
            return enqueue(user);  // capture failed: run the same work directly
        }
        g_graphs.emplace(key, e);
    }
    if (cudaGraphLaunch(e->exec, user) != cudaSuccess) return MOSA_ERR_CUDA;
    replayed(e->rec);
    return MOSA_OK;
}

}  // namespace
}  // namespace mosa

using namespace mosa;

extern "C" {

int32_t mosa_adaptive_k(int32_t T, int32_t rho) {
    if (T < 1 || rho < 1) return 0;
    const int32_t k = T / rho < 2 ? 2 : T / rho;   // Sec. 3.5: max(floor(T / rho), 2)
    return k < T ? k : T;
}

const char *mosa_status_string(mosa_status s) {
    switch (s) {
        case MOSA_OK: return "MOSA_OK";
        case MOSA_ERR_INVALID_ARG: return "MOSA_ERR_INVALID_ARG: invalid argument";
        case MOSA_ERR_UNSUPPORTED: return "MOSA_ERR_UNSUPPORTED: shape outside the supported set";
        case MOSA_ERR_CUDA: return "MOSA_ERR_CUDA: CUDA runtime error";
        case MOSA_ERR_DEVICE_TIMEOUT: return "MOSA_ERR_DEVICE_TIMEOUT: a bounded device wait gave up";
        case MOSA_ERR_WORKSPACE: return "MOSA_ERR_WORKSPACE: workspace missing, misaligned or too small";
        case MOSA_ERR_RANGE:
            return "MOSA_ERR_RANGE: an fp16 attention intermediate (k > 128) exceeded +-65504";
        default: return "unknown mosa_status";
    }
}

size_t mosa_workspace_bytes(const mosa_shape *shape) {
    Dims dm;
    if (check_shape(shape, &dm) != MOSA_OK) return 0;
    return carve(dm, nullptr, nullptr);
}

mosa_status mosa_forward(const mosa_shape *shape, const void *X, const void *W_r,
                         const void *W_q, const void *W_k, const void *W_v, const void *W_o,
                         float *Y, int32_t *I, float *r_sel, float *r_full, void *workspace,
                         size_t workspace_bytes, void *stream) {
    Dims dm;
    mosa_status st = check_shape(shape, &dm);
    if (st != MOSA_OK) return st;
    if (!X || !W_r || !W_q || !W_k || !W_v || !W_o || !Y || !I || !r_sel)
        return MOSA_ERR_INVALID_ARG;
    Saved sv;
    if ((st = check_workspace(dm, workspace, workspace_bytes, &sv)) != MOSA_OK) return st;
    float *rf = r_full ? r_full : sv.r_full;
    DevResources *res = use_tc(dm) ? dev_resources() : nullptr;
    auto enqueue = [&](cudaStream_t s) -> mosa_status {
        return forward_routed(dm, X, W_r, W_q, W_k, W_v, W_o, Y, I, r_sel, rf, sv, s, res);
    };
    const GraphKey key = make_key(0, dm, shape, {X, W_r, W_q, W_k, W_v, W_o, Y, I, r_sel, r_full,
                                                 workspace});
    return run_graphed(key, (cudaStream_t)stream, enqueue);
}

mosa_status mosa_forward_with_indices(const mosa_shape *shape, const void *X, const void *W_q,
                                      const void *W_k, const void *W_v, const void *W_o,
                                      const int32_t *I, const float *r_sel, float *Y,
                                      void *workspace, size_t workspace_bytes, void *stream) {
    Dims dm;
    mosa_status st = check_shape(shape, &dm);
    if (st != MOSA_OK) return st;
    if (!X || !W_q || !W_k || !W_v || !W_o || !I || !r_sel || !Y) return MOSA_ERR_INVALID_ARG;
    Saved sv;
    if ((st = check_workspace(dm, workspace, workspace_bytes, &sv)) != MOSA_OK) return st;
    DevResources *res = use_tc(dm) ? dev_resources() : nullptr;
    auto enqueue = [&](cudaStream_t s) -> mosa_status {
        return forward_given(dm, X, W_q, W_k, W_v, W_o, I, r_sel, Y, sv, s, res);
    };
    const GraphKey key = make_key(1, dm, shape, {X, W_q, W_k, W_v, W_o, I, r_sel, Y, workspace});
    return run_graphed(key, (cudaStream_t)stream, enqueue);
}

mosa_status mosa_backward(const mosa_shape *shape, const void *X, const void *W_r,
                          const void *W_q, const void *W_k, const void *W_v, const void *W_o,
                          const int32_t *I, const float *r_sel, const void *dY, float *dX,
                          float *dW_r, float *dW_q, float *dW_k, float *dW_v, float *dW_o,
                          void *workspace, size_t workspace_bytes, void *stream) {
    Dims dm;
    mosa_status st = check_shape(shape, &dm);
    if (st != MOSA_OK) return st;
    if (!X || !W_r || !W_q || !W_k || !W_v || !W_o || !I || !r_sel || !dY || !dX || !dW_r ||
        !dW_q || !dW_k || !dW_v || !dW_o)
        return MOSA_ERR_INVALID_ARG;
    Saved sv;
    if ((st = check_workspace(dm, workspace, workspace_bytes, &sv)) != MOSA_OK) return st;
    DevResources *res = use_tc(dm) ? dev_resources() : nullptr;
    auto enqueue = [&](cudaStream_t s) -> mosa_status {
        return backward_all(dm, X, W_r, W_q, W_k, W_v, W_o, dY, dX, dW_r, dW_q, dW_k, dW_v, dW_o,
                            sv, s, res);
    };
    const GraphKey key = make_key(2, dm, shape, {X, W_r, W_q, W_k, W_v, W_o, I, r_sel, dY, dX,
                                                 dW_r, dW_q, dW_k, dW_v, dW_o, workspace});
    return run_graphed(key, (cudaStream_t)stream, enqueue);
}

size_t mosa_hybrid_workspace_bytes(const mosa_hybrid_shape *shape) {
    Hybrid h;
    if (check_hybrid(shape, &h) != MOSA_OK) return 0;
    return carve_hybrid(h, nullptr, nullptr);
}

mosa_status mosa_hybrid_forward(const mosa_hybrid_shape *shape, const void *X, const void *W_r,
                                const void *W_q, const void *W_k, const void *W_v,
                                const void *W_o, const void *D_q, const void *D_k,
                                const void *D_v, const void *D_o, float *Y, int32_t *I,
                                float *r_sel, float *r_full, void *workspace,
                                size_t workspace_bytes, void *stream) {
    Hybrid h;
    mosa_status st = check_hybrid(shape, &h);
    if (st != MOSA_OK) return st;
    if (!X || !W_r || !W_q || !W_k || !W_v || !W_o || !Y || !I || !r_sel)
        return MOSA_ERR_INVALID_ARG;
    if (h.has_dense && (!D_q || !D_k || !D_v || !D_o)) return MOSA_ERR_INVALID_ARG;
    HybridSpace sp;
    if ((st = check_hybrid_workspace(h, workspace, workspace_bytes, &sp)) != MOSA_OK) return st;
    float *rf = r_full ? r_full : sp.sparse.r_full;
    DevResources *rs = use_tc(h.sparse) ? dev_resources() : nullptr;
    DevResources *rd = h.has_dense && use_tc(h.dense) ? dev_resources() : nullptr;
    auto enqueue = [&](cudaStream_t s) -> mosa_status {
        mosa_status e = forward_routed(h.sparse, X, W_r, W_q, W_k, W_v, W_o, Y, I, r_sel, rf,
                                       sp.sparse, s, rs);
        if (e != MOSA_OK || !h.has_dense) return e;
        return forward_given(h.dense, X, D_q, D_k, D_v, D_o, nullptr, nullptr, Y, sp.dense, s, rd);
    };
    const GraphKey key = make_key(3, h.sparse, &shape->sparse,
                                  {X, W_r, W_q, W_k, W_v, W_o, D_q, D_k, D_v, D_o, Y, I, r_sel,
                                   r_full, workspace},
                                  h.has_dense ? &h.dense : nullptr, shape->H_dense, shape->window);
    return run_graphed(key, (cudaStream_t)stream, enqueue);
}

mosa_status mosa_hybrid_backward(const mosa_hybrid_shape *shape, const void *X, const void *W_r,
                                 const void *W_q, const void *W_k, const void *W_v,
                                 const void *W_o, const void *D_q, const void *D_k,
                                 const void *D_v, const void *D_o, const int32_t *I,
                                 const float *r_sel, const void *dY, float *dX, float *dW_r,
                                 float *dW_q, float *dW_k, float *dW_v, float *dW_o, float *dD_q,
                                 float *dD_k, float *dD_v, float *dD_o, void *workspace,
                                 size_t workspace_bytes, void *stream) {
    Hybrid h;
    mosa_status st = check_hybrid(shape, &h);
    if (st != MOSA_OK) return st;
    if (!X || !W_r || !W_q || !W_k || !W_v || !W_o || !I || !r_sel || !dY || !dX || !dW_r ||
        !dW_q || !dW_k || !dW_v || !dW_o)
        return MOSA_ERR_INVALID_ARG;
    if (h.has_dense && (!D_q || !D_k || !D_v || !D_o || !dD_q || !dD_k || !dD_v || !dD_o))
        return MOSA_ERR_INVALID_ARG;
    HybridSpace sp;
    if ((st = check_hybrid_workspace(h, workspace, workspace_bytes, &sp)) != MOSA_OK) return st;
    DevResources *rs = use_tc(h.sparse) ? dev_resources() : nullptr;
    DevResources *rd = h.has_dense && use_tc(h.dense) ? dev_resources() : nullptr;
    auto enqueue = [&](cudaStream_t s) -> mosa_status {
        mosa_status e = backward_all(h.sparse, X, W_r, W_q, W_k, W_v, W_o, dY, dX, dW_r, dW_q,
                                     dW_k, dW_v, dW_o, sp.sparse, s, rs);
        if (e != MOSA_OK || !h.has_dense) return e;
        MOSA_TRY(cudaMemsetAsync(sp.zero_wr, 0, sp.zero_wr_bytes, s));
        return backward_all(h.dense, X, sp.zero_wr, D_q, D_k, D_v, D_o, dY, dX, sp.dwr, dD_q,
                            dD_k, dD_v, dD_o, sp.dense, s, rd);
    };
    const GraphKey key = make_key(4, h.sparse, &shape->sparse,
                                  {X, W_r, W_q, W_k, W_v, W_o, D_q, D_k, D_v, D_o, I, r_sel, dY,
                                   dX, dW_r, dW_q, dW_k, dW_v, dW_o, dD_q, dD_k, dD_v, dD_o,
                                   workspace},
                                  h.has_dense ? &h.dense : nullptr, shape->H_dense, shape->window);
    return run_graphed(key, (cudaStream_t)stream, enqueue);
}

mosa_status mosa_topk(int32_t rows, int32_t T, int32_t k, const float *scores, int32_t *I,
                      float *r_sel, void *stream) {
    if (rows <= 0 || T <= 0 || k <= 0 || k > T) return MOSA_ERR_INVALID_ARG;
    if (!scores || !I || !r_sel) return MOSA_ERR_INVALID_ARG;
    if (T > 65536) return MOSA_ERR_UNSUPPORTED;
    return cuda_status(launch_select(rows, T, k, scores, I, r_sel, 0, 1, nullptr, nullptr,
                                     (cudaStream_t)stream));
}

int32_t mosa_stage_engine(const mosa_shape *shape, int32_t stage) {
    Dims dm;
    if (check_shape(shape, &dm) != MOSA_OK || stage < 0 || stage >= kNumStages) return -1;
    switch (stage) {
        case kStageRouter: return (use_tc(dm) && dm.H % 8 == 0) ? 1 : 0;
        case kStageSelect: return 2;
        case kStageQkv:
        case kStageOut:
        case kStageOutBwd:
        case kStageInBwd:
        case kStageWBwd:
        case kStageDwo:
        case kStageAttnFwd:
        case kStageAttnBwd: return use_tc(dm) ? 1 : 0;
        case kStageFwdUnit: return use_fused_forward(dm) ? 1 : 0;
        case kStageBwdUnit: return use_fused_backward(dm) ? 1 : 0;
        default: return 0;
    }
}

int32_t mosa_profile_spans(const mosa_shape *shape, void *workspace, double *ms, int32_t max_stages) {
    Dims dm;
    if (check_shape(shape, &dm) != MOSA_OK || workspace == nullptr || ms == nullptr) return 0;
    Saved sv;
    carve(dm, (char *)workspace, &sv);
    unsigned long long h[2 * 16];
    if (cudaDeviceSynchronize() != cudaSuccess ||
        cudaMemcpy(h, sv.spans, sizeof(h), cudaMemcpyDeviceToHost) != cudaSuccess)
        return 0;
    const int n = max_stages < kNumStages ? max_stages : kNumStages;
    for (int i = 0; i < n; ++i) {
        const unsigned long long a = h[2 * i], b = h[2 * i + 1];
        ms[i] = (a != ~0ull && b != 0ull && b >= a) ? (double)(b - a) * 1e-6 : -1.0;
    }
    return n;
}

mosa_status mosa_profile_spans_copy(const mosa_shape *shape, void *workspace, void *dst,
                                    void *stream) {
    Dims dm;
    mosa_status st = check_shape(shape, &dm);
    if (st != MOSA_OK) return st;
    if (dst == nullptr) return MOSA_ERR_INVALID_ARG;
    if (workspace == nullptr || ((uintptr_t)workspace % kAlign) != 0) return MOSA_ERR_WORKSPACE;
    Saved sv;
    carve(dm, (char *)workspace, &sv);
    return cuda_status(cudaMemcpyAsync(dst, sv.spans, sizeof(unsigned long long) * 2 * 16,
                                       cudaMemcpyDeviceToDevice, (cudaStream_t)stream));
}

int32_t mosa_profile_timeline_read(const mosa_shape *shape, void *workspace, double *start_us,
                                   double *end_us, int32_t max_stages) {
    Dims dm;
    if (check_shape(shape, &dm) != MOSA_OK || workspace == nullptr || start_us == nullptr ||
        end_us == nullptr)
        return 0;
    Saved sv;
    carve(dm, (char *)workspace, &sv);
    unsigned long long h[2 * 16];
    if (cudaDeviceSynchronize() != cudaSuccess ||
        cudaMemcpy(h, sv.spans, sizeof(h), cudaMemcpyDeviceToHost) != cudaSuccess)
        return 0;
    unsigned long long t0 = ~0ull;
    for (int i = 0; i < kNumStages; ++i)
        if (h[2 * i] != ~0ull && h[2 * i + 1] != 0ull && h[2 * i + 1] >= h[2 * i] && h[2 * i] < t0)
            t0 = h[2 * i];
    const int n = max_stages < kNumStages ? max_stages : kNumStages;
    for (int i = 0; i < n; ++i) {
        const unsigned long long a = h[2 * i], b = h[2 * i + 1];
        const bool ok = a != ~0ull && b != 0ull && b >= a && t0 != ~0ull;
        start_us[i] = ok ? (double)(a - t0) * 1e-3 : -1.0;
        end_us[i] = ok ? (double)(b - t0) * 1e-3 : -1.0;
    }
    return n;
}

mosa_status mosa_check_status(const mosa_shape *shape, void *workspace, void *stream) {
    Dims dm;
    mosa_status st = check_shape(shape, &dm);
    if (st != MOSA_OK) return st;
    if (workspace == nullptr || ((uintptr_t)workspace % kAlign) != 0) return MOSA_ERR_WORKSPACE;
    cudaStream_t s = (cudaStream_t)stream;
    uint32_t word = 0;
    if (cudaStreamSynchronize(s) != cudaSuccess) return MOSA_ERR_CUDA;
    if (cudaMemcpy(&word, workspace, sizeof(word), cudaMemcpyDeviceToHost) != cudaSuccess)
        return MOSA_ERR_CUDA;
    if (cudaMemset(workspace, 0, sizeof(word)) != cudaSuccess) return MOSA_ERR_CUDA;
    if (word & kStatusTimeout) return MOSA_ERR_DEVICE_TIMEOUT;
    if (word & kStatusBadIndex) return MOSA_ERR_INVALID_ARG;
    if (word & kStatusRange) return MOSA_ERR_RANGE;
    return MOSA_OK;
}

}  // extern "C"
