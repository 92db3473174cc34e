/*
 * libmosa: Mixture-of-Sparse-Attention (MoSA) layer on one NVIDIA GB300 (sm_103a).
 *
 * The layer (arXiv 2505.00315, Sec. 2.2 and Eq. mosa_mha) for each sequence b
 * and head h:
 *     r      = sigmoid(X[b] W_r[:,h])                 router scores over T tokens
 *     r^topk, I = TopK(r, k)                          k tokens chosen by the head
 *     X^s    = X[b, I, :]                             gathered rows
 *     Q, K, V = X^s W_q[h], X^s W_k[h], X^s W_v[h]
 *     A      = softmax((Q K^T + M) / sqrt(h')) V,     M_ij = 0 iff I_i >= I_j, else -inf
 *     Y[b, I_i, :] += r^topk_i (A W_o[h])_i           scattered back; heads summed
 *
 * Conventions shared by every call:
 *   - All tensor pointers are DEVICE pointers to caller-owned memory; the
 *     layer calls allocate nothing on the device or the host (only the
 *     optional stage timing below creates CUDA events).
 *   - Layouts are dense row-major:
 *       X, dY     [B,T,d]      storage dtype (fp32 or bf16)
 *       W_r       [d,H]        storage dtype
 *       W_q,W_k,W_v [H,d,h']   storage dtype
 *       W_o       [H,h',d]     storage dtype
 *       Y, dX     [B,T,d]      fp32
 *       I         [B,H,k]      int32, strictly ascending token indices
 *       r_sel     [B,H,k]      fp32, r^topk in the order of I
 *       r_full    [B,H,T]      fp32 router scores of every token
 *       dW_r      [d,H]  dW_q,dW_k,dW_v [H,d,h']  dW_o [H,h',d]   fp32
 *   - Calls are asynchronous on `stream` (a cudaStream_t, NULL = legacy default
 *     stream).  They return after argument validation and kernel launch.
 *   - mosa_forward, mosa_forward_with_indices, mosa_backward and the hybrid
 *     calls capture their launch sequence into a CUDA graph the first time
 *     they see a given shape, set of pointers and kernel path, and replay that graph on later
 *     identical calls (one launch instead of about a dozen).  The capture runs
 *     on an internal stream of the current device.  Up to 128 graphs are kept
 *     (driver resources, no user memory); further new calls run unrecorded.
 *     Setting the environment variable MOSA_GRAPHS=0 turns this off.
 *   - Kernel paths (environment, read at every call): MOSA_FORCE_SIMT=1 runs
 *     the CUDA-core kernels only; MOSA_FUSED_FWD=0 runs the k <= 128 forward
 *     as three kernels (projection, attention, output) instead of one fused
 *     kernel; MOSA_FUSED_BWD=1 runs the k <= 128 backward's G, row terms and
 *     attention backward as one fused kernel; MOSA_PDL=0 turns programmatic
 *     dependent launch off; MOSA_HEADSUM=0 turns off the token-major output
 *     product (used for k > 128 when every head keeps at least half of the
 *     tokens) in favour of the row-major one, MOSA_HEADSUM=1 uses the
 *     token-major output and input-gradient products wherever they apply.
 *     All paths compute the same operation.
 *     For tests of the give-up path only: MOSA_TEST_ROUTER_WAIT_NS=n limits
 *     each main-loop wait of the tensor-core router GEMM to n nanoseconds
 *     instead of 2 s (read when the router is launched or captured, so run
 *     such a call with MOSA_GRAPHS=0); a wait that runs out makes
 *     mosa_check_status return MOSA_ERR_DEVICE_TIMEOUT.
 *   - Outputs are overwritten, never accumulated into.
 *   - Arithmetic: fp32 accumulation everywhere.  With bf16 storage the
 *     intermediates fed to tensor-core products are kept as bf16 hi/lo pairs
 *     (v ~ hi + lo, fp32-level accuracy) where they meet the bf16 weights
 *     (the attention output diag(r) A and dQ|dK|dV).  Inside the attention,
 *     Q, K, V, P, dA and dS are pairs too for k <= 128, and single fp16
 *     values (11-bit significand) for k > 128, one MMA per product: a value
 *     beyond the fp16 range (|v| > 65504) is reported as MOSA_ERR_RANGE by
 *     mosa_check_status() rather than passed on silently.  With fp32 storage
 *     every intermediate is fp32.
 *   - Tokens tied on the router score are taken lowest index first.
 *   - NaN inputs give undefined results (but no out-of-bounds access).
 *   - Errors: a call that returns anything but MOSA_OK has launched nothing.
 *     Errors found on the device (invalid caller indices, a bounded wait that
 *     ran out) are recorded in a status word inside the workspace; read and
 *     clear it with mosa_check_status().
 */
#ifndef MOSA_H_
#define MOSA_H_

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
    MOSA_OK = 0,
    MOSA_ERR_INVALID_ARG = 1,     /* bad sizes, NULL pointers, k > T, bad indices */
    MOSA_ERR_UNSUPPORTED = 2,     /* valid but outside what the kernels implement */
    MOSA_ERR_CUDA = 3,            /* a CUDA runtime call or launch failed */
    MOSA_ERR_DEVICE_TIMEOUT = 4,  /* a bounded device-side wait gave up */
    MOSA_ERR_WORKSPACE = 5,       /* workspace NULL, too small or misaligned */
    MOSA_ERR_RANGE = 6            /* an fp16 attention intermediate overflowed (see below) */
} mosa_status;

typedef enum { MOSA_F32 = 0, MOSA_BF16 = 1 } mosa_dtype;

/* Problem size.  B sequences of T tokens of width d; H MoSA heads of size hp
 * (the paper's h'); each head keeps k of the T tokens (Sec. 2.2).
 * first_token = 1 makes every head keep token 0 of each sequence and select
 * the other k-1 tokens by router score among tokens 1..T-1 (the IsoFLOP
 * models of Sec. 3.2); token 0 is scaled by its own router score like the
 * others.  first_token = 0 is the plain TopK; other values are invalid. */
typedef struct {
    int32_t B, T, d, H, hp, k;
    int32_t dtype;       /* mosa_dtype of X, dY and all weights */
    int32_t first_token; /* 0 or 1, see above */
    int32_t rope;        /* 0 or 1: rotary position encoding, see below */
} mosa_shape;
/* rope = 1 rotates each head's queries and keys after the projections by the
 * tokens' original positions t = I[b,h,i] (Sec. 2.2, positional encodings):
 * pair (2p, 2p+1) of the first h'/2 dimensions turns by t * 10000^(-2p/(h'/2)),
 * the other h'/2 dimensions are left unchanged.  A backward must be given the
 * same rope value as its forward. */

/* Supported sizes (else MOSA_ERR_UNSUPPORTED):
 *   1 <= k <= T <= 65536; B, H >= 1; B*T*d < 2^31; H*d*hp < 2^31;
 *   d % 8 == 0 and hp in {16, 32, 64, 128}. */

/* Tokens per head for a sequence of T tokens at sparsity rho (Sec. 3.5, for
 * inputs shorter than the training length): k = max(floor(T / rho), 2),
 * and at most T.  Returns 0 if T < 1 or rho < 1. */
int32_t mosa_adaptive_k(int32_t T, int32_t rho);

/* Human-readable name of a status code (static string, never NULL). */
const char *mosa_status_string(mosa_status s);

/* Bytes of device workspace the calls below need for `shape`; 0 if the shape
 * is invalid or unsupported.  The workspace carries the state that
 * mosa_backward reuses from mosa_forward (router scores, selected rows,
 * Q/K/V, attention output and its log-sum-exp) plus the status word, so the
 * same buffer must be passed to a forward and the backward that follows it.
 * It must be 256-byte aligned. */
size_t mosa_workspace_bytes(const mosa_shape *shape);

/* Forward pass of the layer (Sec. 2.2, Eq. mosa_mha): router, TopK, gather,
 * per-head projections, index-masked causal attention, diag(r^topk) A W_o and
 * the scatter-sum into Y.
 *   X, W_r, W_q, W_k, W_v, W_o : inputs (storage dtype), see layouts above.
 *   Y      : [B,T,d] fp32 output; rows chosen by no head are 0.
 *   I      : [B,H,k] int32 output, ascending.
 *   r_sel  : [B,H,k] fp32 output, r at I.
 *   r_full : [B,H,T] fp32 output of all router scores, or NULL.
 *   workspace, workspace_bytes : see mosa_workspace_bytes.
 *   stream : cudaStream_t.
 * Returns MOSA_OK, MOSA_ERR_INVALID_ARG, MOSA_ERR_UNSUPPORTED,
 * MOSA_ERR_WORKSPACE or MOSA_ERR_CUDA. */
mosa_status mosa_forward(const mosa_shape *shape, const void *X, const void *W_r,
                         const void *W_q, const void *W_k, const void *W_v, const void *W_o,
                         float *Y, int32_t *I, float *r_sel, float *r_full, void *workspace,
                         size_t workspace_bytes, void *stream);

/* Forward pass with caller-chosen token sets (no router, no TopK): the
 * fixed-sparse special case of Sec. 3.1 (I = [0, rho, 2rho, ...], r = 1) and
 * any other externally routed variant.
 *   I     : [B,H,k] int32 input, strictly ascending and in [0,T) per row.
 *           Rows breaking this are replaced by 0..k-1 and flagged in the
 *           status word (MOSA_ERR_INVALID_ARG from mosa_check_status).
 *   r_sel : [B,H,k] fp32 input scores applied as diag(r_sel).
 *   Y     : [B,T,d] fp32 output.
 * W_r is not read.  The workspace afterwards holds the state mosa_backward
 * needs, but the router gradient it then reports assumes r_sel =
 * sigmoid(X W_r)[I]. */
mosa_status mosa_forward_with_indices(const mosa_shape *shape, const void *X,
                                      const void *W_q, const void *W_k, const void *W_v,
                                      const void *W_o, const int32_t *I, const float *r_sel,
                                      float *Y, void *workspace, size_t workspace_bytes,
                                      void *stream);

/* Backward pass: gradients of <Y, dY> with the token sets held constant
 * (TopK is not differentiated; the router learns through the diag(r^topk)
 * scaling only, Sec. 2.2).  Must follow a mosa_forward (or
 * mosa_forward_with_indices) on the same stream, with the same shape, inputs
 * and workspace; I and r_sel are that call's outputs.
 *   dY : [B,T,d] upstream gradient (storage dtype).
 *   dX [B,T,d], dW_r [d,H], dW_q/dW_k/dW_v [H,d,hp], dW_o [H,hp,d] : fp32 outputs.
 * Returns as mosa_forward. */
mosa_status mosa_backward(const mosa_shape *shape, const void *X, const void *W_r,
                          const void *W_q, const void *W_k, const void *W_v, const void *W_o,
                          const int32_t *I, const float *r_sel, const void *dY, float *dX,
                          float *dW_r, float *dW_q, float *dW_k, float *dW_v, float *dW_o,
                          void *workspace, size_t workspace_bytes, void *stream);

/* Hybrid layer (Sec. 2.2, hybridization; Sec. 3.4): the MoSA heads of
 * `sparse` plus H_dense dense heads, all summed into one Y (Eq. mha).  A
 * dense head attends causally over all T tokens with no router and no
 * scaling (Sec. 2.1).  window = w > 0 makes them local heads for long
 * sequences (Sec. 3.4): token i sees token j iff j <= i and both lie in the
 * same block of w positions (the block pattern of fixed sparse attention;
 * T % w == 0, else MOSA_ERR_UNSUPPORTED).  window = 0 (or T) is the dense
 * case.  Dense and local heads use the head size hp, the dtype and the rope
 * setting of `sparse` (positions 0..T-1); first_token applies to the MoSA
 * heads only.  H_dense = 0 is a plain MoSA layer. */
typedef struct {
    mosa_shape sparse;  /* the MoSA heads */
    int32_t H_dense;    /* >= 0 */
    int32_t window;     /* 0 <= window <= T */
} mosa_hybrid_shape;

/* Workspace bytes of a hybrid forward and its backward; 0 if the shape is
 * invalid or unsupported.  256-byte aligned, as for mosa_workspace_bytes;
 * mosa_check_status(&shape->sparse, workspace, stream) reports for both
 * head groups. */
size_t mosa_hybrid_workspace_bytes(const mosa_hybrid_shape *shape);

/* Forward of the hybrid layer.  Arguments as mosa_forward, plus the dense
 * heads' weights D_q, D_k, D_v [H_dense,d,hp] and D_o [H_dense,hp,d] in the
 * storage dtype (may be NULL when H_dense = 0).  Y [B,T,d] fp32 is
 * overwritten with the sum of both head groups; I, r_sel, r_full are the MoSA
 * heads'.  Returns as mosa_forward. */
mosa_status mosa_hybrid_forward(const mosa_hybrid_shape *shape, const void *X, const void *W_r,
                                const void *W_q, const void *W_k, const void *W_v,
                                const void *W_o, const void *D_q, const void *D_k,
                                const void *D_v, const void *D_o, float *Y, int32_t *I,
                                float *r_sel, float *r_full, void *workspace,
                                size_t workspace_bytes, void *stream);

/* Backward of the hybrid layer; must follow mosa_hybrid_forward on the same
 * stream with the same shape, inputs and workspace.  dX [B,T,d] receives the
 * sum over both head groups; dW_r .. dW_o are the MoSA heads' gradients (as
 * mosa_backward), dD_q, dD_k, dD_v [H_dense,d,hp] and dD_o [H_dense,hp,d] the
 * dense heads' (fp32, overwritten).  Returns as mosa_backward. */
mosa_status mosa_hybrid_backward(const mosa_hybrid_shape *shape, const void *X, const void *W_r,
                                 const void *W_q, const void *W_k, const void *W_v,
                                 const void *W_o, const void *D_q, const void *D_k,
                                 const void *D_v, const void *D_o, const int32_t *I,
                                 const float *r_sel, const void *dY, float *dX, float *dW_r,
                                 float *dW_q, float *dW_k, float *dW_v, float *dW_o, float *dD_q,
                                 float *dD_k, float *dD_v, float *dD_o, void *workspace,
                                 size_t workspace_bytes, void *stream);

/* TopK alone (Sec. 2.2): for each of `rows` rows of T fp32 scores, the k
 * largest (ties: lower index first), written ascending by index.
 *   scores [rows,T] fp32 input; I [rows,k] int32 and r_sel [rows,k] fp32 outputs.
 * Needs no workspace.  1 <= k <= T <= 65536.  Scores must not be NaN. */
mosa_status mosa_topk(int32_t rows, int32_t T, int32_t k, const float *scores, int32_t *I,
                      float *r_sel, void *stream);

/* Waits for `stream`, then reads and clears the device status word in the
 * workspace: MOSA_OK, MOSA_ERR_INVALID_ARG (caller indices were invalid),
 * MOSA_ERR_DEVICE_TIMEOUT or MOSA_ERR_RANGE (an fp16 intermediate of the
 * k > 128 attention overflowed; the outputs are then not valid); MOSA_ERR_CUDA
 * if the wait itself failed. */
mosa_status mosa_check_status(const mosa_shape *shape, void *workspace, void *stream);


/* Routing without a workspace: router scores r = sigmoid(X W_r) and TopK, the
 * same I and r_sel as mosa_forward, for callers that cannot allocate device
 * memory.  The paper has no counterpart; this exists for callers whose
 * device heap belongs to someone else (a host application that hands out no
 * buffers after start-up, a plug-in interface that passes only inputs and
 * outputs) or that must never pay cudaMalloc's implicit synchronisation.
 * It allocates nothing: the [B,H,T] scores live in a 4 MiB array compiled
 * into the library (held on every GPU that loads it until the process
 * exits), so B*H*T may be at most 1,048,576 (else MOSA_ERR_UNSUPPORTED).
 *   X [B,T,d], W_r [d,H] : inputs (storage dtype); hp is validated but unused.
 *   I [B,H,k] int32, r_sel [B,H,k] fp32 : outputs, as mosa_forward (the same
 *   router kernel computes the scores, so the results are identical).
 * Every call looks up the array's device address on the current device (the
 * host-side symbol is not a device address); the first call on a device also
 * loads the library's device code there, so make it before any stream
 * capture.  After a cudaDeviceReset the next call finds the array anew.
 * All calls share the one array and the contents of the last call remain in
 * it; nothing needs clearing, because each call writes every score it reads.
 * Calls whose GPU work overlaps (different streams or host threads without
 * ordering) race on the array: order them on one stream.  There is no status
 * word: a bounded device wait that runs out leaves I and r_sel undefined.
 * Returns MOSA_OK, MOSA_ERR_INVALID_ARG, MOSA_ERR_UNSUPPORTED or MOSA_ERR_CUDA. */
mosa_status mosa_route_noalloc(const mosa_shape *shape, const void *X, const void *W_r,
                               int32_t *I, float *r_sel, void *stream);

/* ---- Measurement support (not part of the layer) ----------------------
 * Stages: 0 router, 1 select, 2 qkv, 3 attn_fwd, 4 out, 5 out_bwd,
 * 6 attn_bwd, 7 in_bwd, 8 w_bwd, 9 dwo (dW_o), 10 fwd_unit (F3-F5 fused,
 * k <= 128), 11 bwd_unit (G, row terms and attention backward fused, k <= 128,
 * opt-in).  A hybrid call times each stage once per head group.  These calls
 * create CUDA events (host-side handles, no device memory) when stage timing
 * is on. */

/* Number of kernels this library has launched since it was loaded. */
unsigned long long mosa_kernel_launches(void);

/* Turns CUDA-event timing on for the stages whose bit is set in stage_mask
 * (0 turns it off).  Each timed stage of later calls records an event pair on
 * the call's stream.  Always MOSA_OK. */
mosa_status mosa_profile_stages(uint32_t stage_mask);

/* Waits for the recorded events, writes per stage the summed elapsed
 * milliseconds and the number of timed launches (arrays of max_stages
 * entries, either may be NULL), resets the sums and returns the number of
 * stages the library has. */
int32_t mosa_profile_read(double *total_ms, int32_t *count, int32_t max_stages);

/* Device time of the stages timed by the last layer call with this
 * workspace: for each stage (ms[0 .. max_stages-1]), the span in
 * milliseconds from the first CTA start to the last CTA end of its
 * tensor-core and selection kernels (%globaltimer stamps written into the
 * workspace while the stage's timing is on), or -1 if it recorded none.
 * Unlike the event timing above, this excludes the time a stage's kernels
 * wait for a launch or for SMs before they start.  Waits for the device.
 * Returns the number of entries written. */
int32_t mosa_profile_spans(const mosa_shape *shape, void *workspace, double *ms, int32_t max_stages);

/* Enqueues on `stream` a device-to-device copy of the workspace's kernel-span
 * slots (32 unsigned 64-bit values: start, end in %globaltimer nanoseconds
 * for stages 0..15; a start of all ones or an end of 0 means no record) into
 * dst (device memory of 256 bytes), so that a caller timing many steps can
 * keep each step's spans without waiting for the device between steps.  The
 * slots are those mosa_profile_spans reads.  MOSA_OK, MOSA_ERR_INVALID_ARG,
 * MOSA_ERR_WORKSPACE or MOSA_ERR_CUDA. */
mosa_status mosa_profile_spans_copy(const mosa_shape *shape, void *workspace, void *dst,
                                    void *stream);

/* Timeline mode (on = 1, off = 0): later layer calls record, for every stage,
 * the first CTA start and last CTA end of its kernels (%globaltimer) into the
 * workspace, with no CUDA events and no per-stage resets between the kernels
 * (which would break the early-launch chain the timing is meant to show);
 * each call instead starts with one small kernel that clears its stages'
 * slots.  Read with mosa_profile_timeline_read.  MOSA_OK, or
 * MOSA_ERR_INVALID_ARG for another value of on. */
mosa_status mosa_profile_timeline(int32_t on);

/* The timeline left in the workspace by the last forward and backward calls
 * with it: start_us[i] and end_us[i] (arrays of max_stages entries) in
 * microseconds from the earliest recorded start, -1 for a stage with no
 * record.  Waits for the device.  Returns the number of entries written, 0 on
 * an invalid shape or pointer or a CUDA error. */
int32_t mosa_profile_timeline_read(const mosa_shape *shape, void *workspace, double *start_us,
                                   double *end_us, int32_t max_stages);

/* Name of a stage ("router", "select", ...; "unknown" if out of range). */
const char *mosa_stage_name(int32_t stage);

/* Which units the kernels of `stage` run on for `shape`, so that a timing can
 * be set against the right roofline: 0 CUDA cores (fp32 FFMA), 1 tensor cores
 * (tcgen05), 2 memory-bound data movement; -1 for an invalid shape or stage. */
int32_t mosa_stage_engine(const mosa_shape *shape, int32_t stage);

#ifdef __cplusplus
}
#endif
#endif /* MOSA_H_ */
