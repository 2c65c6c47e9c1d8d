/*
 * omq.h — C ABI of libomq: one OmniQuant block-calibration step on a GB300 (sm_103a).
 *
 * The step is the inner loop of Algorithm 1 (Appendix A): apply the learnable
 * equivalent transformation (LET, Eq. 3-5) and learnable weight clipping (LWC,
 * Eq. 2) to a transformer block, run the quantized block on a calibration sample,
 * take the MSE against the full-precision block output (Eq. 1), and back-propagate
 * with the straight-through estimator to gamma, beta (Theta1) and s, delta, s_a
 * (Theta2).
 *
 * Conventions shared by every entry point
 * ---------------------------------------
 *  - Memory: every tensor pointer is a DEVICE pointer owned by the caller.  The
 *    library never allocates, frees or synchronises; every call only enqueues
 *    work on `stream` and returns.  Scratch memory is a caller-provided workspace
 *    whose size is queried first.
 *  - Layouts are row-major.  A weight W is [Cout, Cin] (the transpose of the
 *    paper's C_in x C_out notation in Sec. 3.3); activations are [T, C].
 *  - Dtypes: frozen weights bf16; activations, learnable parameters, per-group /
 *    per-token scales and all gradients fp32; zero points and argmax/argmin
 *    indices int32; integer codes uint8.
 *  - Alignment: every pointer must be 16-byte aligned and every inner dimension a
 *    multiple of 8 elements, else OMQ_ERR_ALIGN.  There is no slow path.
 *  - Errors: argument errors are found on the host before any launch, and then
 *    nothing is written.  Device-side failures (a bounded wait that expired) are
 *    written to the optional `dev_status` word of omq_qcfg and read back with
 *    omq_stream_status.  The library never aborts, traps or prints.
 *  - Gradient outputs are overwritten unless cfg->accumulate is 1, in which case
 *    they are added to.
 *  - Rounding: round() of Eq. 2 is round-half-to-even; every matrix-product operand
 *    is rounded to bf16 (nearest-even) and accumulated in fp32.
 */
#ifndef OMQ_H
#define OMQ_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef struct CUstream_st* omq_stream_t;   /* same type as cudaStream_t; NULL = legacy default stream */

typedef enum {
  OMQ_OK = 0,
  OMQ_ERR_INVALID_ARG = 1,   /* null where required, bad enum value */
  OMQ_ERR_SHAPE = 2,         /* zero or negative size, group does not divide Cin, heads do not divide */
  OMQ_ERR_ALIGN = 3,         /* pointer not 16-byte aligned or inner dimension not a multiple of 8 */
  OMQ_ERR_UNSUPPORTED = 4,   /* bit width outside [2, 8] (or 16 = off); device is not sm_103 */
  OMQ_ERR_CUDA = 5,          /* a launch failed */
  OMQ_ERR_TIMEOUT = 6,       /* a device-side bounded wait expired (reported through dev_status) */
  OMQ_ERR_WORKSPACE = 7      /* workspace smaller than the queried size */
} omq_status;

/* Quantization configuration (Sec. 4.1 "Quantization"). */
typedef struct {
  int32_t wbits;       /* weight bits N of Eq. 2: 2..8, or 16 = weights not quantized            */
  int32_t abits;       /* per-token activation bits: 2..8, or 16 = activations not quantized     */
  int32_t group;       /* weight group size along Cin; 0 = one group per output channel          */
  int32_t let;         /* 1 = learnable equivalent transformation on (Eq. 3, Eq. 5)               */
  float   h_eps;       /* floor of the quantizer step h (1e-5); a floored h has zero gradient    */
  int32_t accumulate;  /* 1 = add into gradient outputs instead of overwriting them              */
  int32_t* dev_status; /* optional device int32: 0 = ok, else an omq_status set by a kernel      */
  int32_t pbits;       /* softmax-output bits (the ablation beside Table A7): 2..8, or 0 / 16 = the
                          softmax output is not quantized (the method's default)                  */
  int32_t wprep;       /* block step / forward only, where the weights are quantized: how the q|k|v
                          products get W_hat (Eq. 2).  0 = the LWC forward writes W_hat (bf16) to
                          HBM and the forward and dX products read it; 1 = both products read the
                          raw bf16 weight and fake-quantize each tile in shared memory with the
                          quantizer state the LWC forward wrote (W_hat never reaches HBM).  The two
                          give bit-identical results; other entry points ignore the field.        */
} omq_qcfg;

/* ------------------------------------------------------------------------------------------
 * Kernel-level entry points
 * ------------------------------------------------------------------------------------------ */

/* Eq. 3.  X~ = (X - delta) / s per input channel, W~ = W diag(s), B~ = B + W delta.
 *   X [T, Cin] fp32, W [Cout, Cin] bf16, B [Cout] fp32 or NULL (= 0), s, delta [Cin] fp32.
 *   Xt [T, Cin] fp32 (NULL = skip), Wt [Cout, Cin] fp32 (NULL = skip), Bt [Cout] fp32 (NULL = skip). */
omq_status omq_let_apply(omq_stream_t stream, int64_t T, int64_t Cin, int64_t Cout,
                         const float* X, const void* W, const float* B, const float* s,
                         const float* delta, float* Xt, float* Wt, float* Bt, const omq_qcfg* cfg);

/* Eq. 2 (LWC) on W~ = r_o * W_oi * s_i, per group of cfg->group input channels of one output row.
 *   W [Cout, Cin] bf16; s [Cin] (NULL = 1: LET scale of Eq. 3); r [Cout] (NULL = 1: row scale, the
 *   1/s_o that the [v, out] LET pair puts on v_proj's rows).  gamma_logit, beta_logit
 *   [Cout, ngroups] fp32 with gamma = sigmoid(gamma_logit).
 *   Outputs: Wq [Cout, Cin] bf16 fake-quantized value (q - z) h (NULL = skip); codes [Cout, Cin]
 *   uint8 (NULL = skip); h [Cout, ngroups] fp32; z int32; argmax / argmin int32 = column index
 *   (in 0..Cin-1) of the first max / min of each group.
 *   bias_delta [Cin] (NULL = skip) and bias_shift [Cout] (NULL = 0): when bias_delta is given, also
 *   writes Bt[o] = r_o * (sum_i W_oi bias_delta_i - bias_shift_o) (the B~ of Eq. 3). */
omq_status omq_lwc_fakequant_fwd(omq_stream_t stream, int64_t Cout, int64_t Cin, const void* W,
                                 const float* s, const float* r, const float* gamma_logit,
                                 const float* beta_logit, void* Wq, uint8_t* codes, float* h,
                                 int32_t* z, int32_t* argmax, int32_t* argmin,
                                 const float* bias_delta, const float* bias_shift, float* Bt,
                                 const omq_qcfg* cfg);

/* Straight-through backward of omq_lwc_fakequant_fwd, given dWq = dL/dWq [Cout, Cin] fp32 and the
 * saved h, z, argmax, argmin.  Every round() has derivative 1; clamp passes the gradient for
 * 0 <= code <= 2^N-1; max/min route theirs to the saved first index; h is not detached.
 *   dgamma, dbeta [Cout, ngroups] fp32.  dWt [Cout, Cin] fp32 = dL/dW~ (NULL = skip).
 *   ds [Cin] (NULL = skip) = sum_o dWt_oi W_oi r_o;  dr [Cout] (NULL = skip) = sum_i dWt_oi W_oi s_i.
 *   dBt [Cout] (NULL = none) with ddelta [Cin] (NULL = skip): ddelta_i = sum_o dBt_o r_o W_oi, the
 *   bias path of Eq. 3.  A scratch workspace of omq_lwc_bwd_workspace_size bytes is required when
 *   ds or ddelta is requested. */
omq_status omq_lwc_fakequant_bwd(omq_stream_t stream, int64_t Cout, int64_t Cin, const void* W,
                                 const float* s, const float* r, const float* gamma_logit,
                                 const float* beta_logit, const float* h, const int32_t* z,
                                 const int32_t* argmax, const int32_t* argmin, const float* dWq,
                                 float* dgamma, float* dbeta, float* dWt, float* ds, float* dr,
                                 const float* dBt, float* ddelta, void* workspace, size_t ws_bytes,
                                 const omq_qcfg* cfg);
size_t omq_lwc_bwd_workspace_size(int64_t Cout, int64_t Cin);

/* LET on activations (Eq. 3, X~ = (X - delta)/s; s, delta NULL = identity) followed by Q_a, the
 * per-token MinMax quantizer (Eq. 2 with gamma = beta = 1, one group per row, N = cfg->abits).
 *   X [T, C] fp32 -> Xq [T, C] bf16 = (q - z) h (or bf16(X~) when abits = 16);
 *   codes [T, C] uint8 (NULL = skip); h [T] fp32, z [T], argmax [T], argmin [T] int32
 *   (all NULL allowed when abits = 16). */
omq_status omq_act_quant_per_token(omq_stream_t stream, int64_t T, int64_t C, const float* X,
                                   const float* s, const float* delta, void* Xq, uint8_t* codes,
                                   float* h, int32_t* z, int32_t* argmax, int32_t* argmin,
                                   const omq_qcfg* cfg);

/* Straight-through backward of omq_act_quant_per_token, given dXq [T, C] fp32 and the saved
 * per-token state.  dX [T, C] fp32 = dL/dX; ds, ddelta [C] (NULL = skip) are the LET column sums
 * ds_i = -sum_t dX~_ti X~_ti / s_i and ddelta_i = -sum_t dX~_ti / s_i.  Needs a workspace of
 * omq_act_bwd_workspace_size bytes when ds or ddelta is requested. */
omq_status omq_act_quant_per_token_bwd(omq_stream_t stream, int64_t T, int64_t C, const float* X,
                                       const float* s, const float* delta, const float* h,
                                       const int32_t* z, const int32_t* argmax,
                                       const int32_t* argmin, const float* dXq, float* dX,
                                       float* ds, float* ddelta, void* workspace, size_t ws_bytes,
                                       const omq_qcfg* cfg);
size_t omq_act_bwd_workspace_size(int64_t T, int64_t C);

/* Block loss of Eq. 1 / Algorithm 1, read as the mean over the n elements of (Yq - Yfp)^2.
 *   loss: device fp32 scalar (overwritten).  dY [n] fp32 = 2 (Yq - Yfp) / n (NULL = skip);
 *   dY_bf16 [n] bf16 copy of dY (NULL = skip).  Needs omq_loss_workspace_size bytes. */
omq_status omq_block_loss(omq_stream_t stream, int64_t n, const float* Yq, const float* Yfp,
                          float* loss, float* dY, void* dY_bf16, void* workspace, size_t ws_bytes);
size_t omq_loss_workspace_size(int64_t n);

/* omq_block_loss for callers that cannot allocate device memory: code whose device memory belongs
 * to another framework's fixed arena, interfaces that pass only inputs and outputs, and code that
 * must not call cudaMalloc/cudaFree (which can synchronize the device) while work is in flight.
 * The paper has no counterpart; it computes exactly what omq_block_loss computes.
 *   Scratch: the partial sums live in a file-scope device array of 1024 floats (4 KB) that every
 *   GPU which loads the library holds until the process exits.  No workspace argument, and no
 *   cudaMalloc, cudaFree or allocating routine of any library is called.
 *   Limit: 1 <= n <= OMQ_NOALLOC_LOSS_MAX_N; other sizes return OMQ_ERR_SHAPE before any launch.
 *   Set-up: a call looks up the array's device address on the current device with
 *   cudaGetSymbolAddress whenever its stream is not being captured (so a device reset, which
 *   reloads the module, leaves no stale address) and otherwise reuses the address of the last
 *   lookup; make the first call on a device before any stream capture.
 *   Sharing: all calls on a device share the array and it keeps the last call's contents; each
 *   call writes every partial it later reads, so nothing needs clearing.  Calls that overlap on
 *   the GPU (different streams without ordering) race on the array: order them. */
#define OMQ_NOALLOC_LOSS_MAX_N 2147483647LL
omq_status omq_block_loss_noalloc(omq_stream_t stream, int64_t n, const float* Yq, const float* Yfp,
                                  float* loss, float* dY, void* dY_bf16);

/* Dense bf16 tensor-core matrix product used by every linear and attention product:
 *   C[b, m, n] = alpha * sum_k A[b, m, k] B[b, n, k] (+ bias[n]) (+ R[b, m, n]) (+ beta_acc * C)
 * A element (b, m, k) is at A + b*a_bs + (a_kmajor ? m*a_ld + k : k*a_ld + m); B likewise with n.
 * Operands bf16, accumulation fp32 in tensor memory (tcgen05).  Cf [b, m, n] fp32 at
 * Cf + b*c_bs + m*ldc + n (NULL = skip); Cb the same positions in bf16 (NULL = skip).
 * causal: 0 none; 1 = skip output tiles with n-start > m-end (scores); 2 = k < m-tile end only
 * (P V, dS K); 3 = k >= m-tile start only (P^T dO, dS^T Q).  Causal tiles assume square 128 tiles. */
omq_status omq_gemm_bf16(omq_stream_t stream, int64_t M, int64_t N, int64_t K, int64_t batch,
                         const void* A, int64_t a_ld, int64_t a_bs, int32_t a_kmajor,
                         const void* B, int64_t b_ld, int64_t b_bs, int32_t b_kmajor,
                         float* Cf, void* Cb, int64_t ldc, int64_t c_bs, float alpha,
                         const float* bias, const float* R, int64_t ldr, float beta_acc,
                         int32_t causal, int32_t* dev_status);

/* Failure-detection self-test (the paper has no counterpart): checks that a device-side wait
 * that never completes ends with OMQ_ERR_TIMEOUT instead of a hang.  Runs the tensor-core product
 * of omq_gemm_bf16, C [M, N] fp32 = A [M, K] B [N, K]^T (bf16, both K-major, rows packed; one
 * CTA: M <= 128, N <= 128, K <= 8192, N and K multiples of 8), with every mbarrier wait bounded
 * by wait_limit_ns (1e3 .. 1e9) instead of the library's one second.  withhold = 1: the first
 * operand load is never issued, so the wait for it expires; the kernel then writes
 * OMQ_ERR_TIMEOUT to *dev_status (if it is still 0), waits (bounded) for the loads it did issue,
 * releases its tensor memory and returns, leaving C unspecified.  withhold = 0: an ordinary
 * product.  The return value covers the launch only; read *dev_status with omq_stream_status. */
omq_status omq_selftest_bounded_wait(omq_stream_t stream, int64_t M, int64_t N, int64_t K, const void* A,
                                     const void* B, float* C, uint64_t wait_limit_ns, int32_t withhold,
                                     int32_t* dev_status);

/* ------------------------------------------------------------------------------------------
 * Single quantized linear (Eq. 4): Y = Q_a(X~) Q_w(W~)^T + B~, and its STE backward.
 * ------------------------------------------------------------------------------------------ */
typedef struct {
  void*    w_hat;   /* [Cout, Cin] bf16 fake-quantized W~                                    */
  float*   h_w;     /* [Cout, ngroups] */
  int32_t* z_w;
  int32_t* imax_w;
  int32_t* imin_w;
  void*    x_hat;   /* [T, Cin] bf16 quantized (or rounded) X~                               */
  float*   h_a;     /* [T] (unused when abits = 16) */
  int32_t* z_a;
  int32_t* imax_a;
  int32_t* imin_a;
  float*   b_tilde; /* [Cout] fp32 B~ */
} omq_qlinear_saved;

omq_status omq_qlinear_fwd(omq_stream_t stream, int64_t T, int64_t Cin, int64_t Cout,
                           const float* X, const void* W, const float* B, const float* s,
                           const float* delta, const float* gamma_logit, const float* beta_logit,
                           float* Y, const omq_qlinear_saved* saved, const omq_qcfg* cfg);
/* dY [T, Cout] fp32.  dX [T, Cin] fp32 (NULL = skip).  dgamma, dbeta [Cout, ngroups];
 * ds, ddelta [Cin] (required when cfg->let). */
omq_status omq_qlinear_bwd(omq_stream_t stream, int64_t T, int64_t Cin, int64_t Cout,
                           const float* X, const void* W, const float* s, const float* delta,
                           const float* gamma_logit, const float* beta_logit,
                           const omq_qlinear_saved* saved, const float* dY, float* dX,
                           float* dgamma, float* dbeta, float* ds, float* ddelta,
                           void* workspace, size_t ws_bytes, const omq_qcfg* cfg);
size_t omq_qlinear_workspace_size(int64_t T, int64_t Cin, int64_t Cout, const omq_qcfg* cfg);
/* Element counts of the omq_qlinear_saved arrays, in the struct's field order (w_hat, h_w, z_w,
 * imax_w, imin_w, x_hat, h_a, z_a, imax_a, imin_a, b_tilde), written to sizes[0..10] (host array
 * owned by the caller); the caller allocates each array with its field's element type (bf16, fp32
 * or int32).  Pure host function.  OMQ_ERR_SHAPE for non-positive sizes or a group that does not
 * divide Cin; the configuration checks of omq_check_cfg otherwise. */
omq_status omq_qlinear_saved_sizes(int64_t T, int64_t Cin, int64_t Cout, const omq_qcfg* cfg, int64_t* sizes);

/* ------------------------------------------------------------------------------------------
 * One LLaMA decoder block (RMSNorm -> RoPE causal attention -> RMSNorm -> SwiGLU FFN), the
 * block F of Eq. 1.  LET pairs (Sec. 3.3 and the appendix ablation of LET positions):
 * [ln1, (q, k, v)] with s1, d1 [d]; [v, out] with so, do [n_kv*hd] moved into v_proj;
 * [Q, K] with sa [n_kv*hd] applied after RoPE; [ln2, (gate, up)] with s2, d2 [d]; none on down.
 * With grouped KV heads so, do, sa are broadcast to the query heads of each group.
 * ------------------------------------------------------------------------------------------ */
typedef struct {
  int32_t T;          /* tokens of one calibration sample */
  int32_t d;          /* hidden size */
  int32_t n_heads;    /* query heads */
  int32_t n_kv;       /* key/value heads (divides n_heads) */
  int32_t head_dim;   /* must be 128 */
  int32_t ffn;        /* SwiGLU inner size */
  float   rms_eps;
  float   rope_theta;
} omq_block_shape;

/* Frozen bf16 weights, [Cout, Cin].  wqkv stacks the rows of q_proj [n_heads*hd, d], k_proj
 * [n_kv*hd, d] and v_proj [n_kv*hd, d]; wgu stacks gate_proj [ffn, d] then up_proj [ffn, d]. */
typedef struct {
  const void* wqkv;
  const void* wo;     /* [d, n_heads*hd] */
  const void* wgu;
  const void* wd;     /* [d, ffn] */
} omq_block_weights;

/* LWC logits [Cout, ngroups] fp32 stacked like the weights, and the LET vectors (NULL when
 * cfg->let = 0).  The gradient struct has the same layout. */
typedef struct {
  float* gamma_qkv; float* beta_qkv;
  float* gamma_o;   float* beta_o;
  float* gamma_gu;  float* beta_gu;
  float* gamma_d;   float* beta_d;
  float* s1; float* d1;   /* [d] */
  float* so; float* do_;  /* [n_kv*hd] */
  float* sa;              /* [n_kv*hd] */
  float* s2; float* d2;   /* [d] */
} omq_block_params;

size_t omq_block_workspace_size(const omq_block_shape* shape, const omq_qcfg* cfg);

/* Forward of the quantized block on x [T, d] fp32 (y [T, d] fp32 out).  With wbits = abits = 16
 * and let = 0 this is the full-precision block that produces the Eq. 1 target. */
omq_status omq_block_forward(omq_stream_t stream, const omq_block_shape* shape,
                             const omq_block_weights* w, const omq_block_params* theta,
                             const float* x, float* y, void* workspace, size_t ws_bytes,
                             const omq_qcfg* cfg);

/* One calibration step without the parameter update: forward, loss = mean((y - y_fp)^2) written
 * to the device scalar `loss`, and the STE gradients of every learnable parameter into `grads`.
 * y (NULL = not returned) receives the quantized block output.
 * The launches go to `stream` and to one auxiliary stream per device owned by the library, joined
 * back to `stream` by events before the call returns, so the call can be captured into a CUDA
 * graph on `stream`.  The library keeps no state keyed on the caller's pointers; a captured graph
 * does: it replays the addresses it was captured with.  A caller that replays (the package's
 * BlockState looks its graphs up by the addresses of x and y_fp) refills the same buffers in place
 * between replays and keeps them alive; new buffers need a new capture. */
omq_status omq_block_step(omq_stream_t stream, const omq_block_shape* shape,
                          const omq_block_weights* w, const omq_block_params* theta,
                          const float* x, const float* y_fp, float* y, float* loss,
                          const omq_block_params* grads, void* workspace, size_t ws_bytes,
                          const omq_qcfg* cfg);

/* Where omq_block_forward / omq_block_step keep the block's stage values inside the caller's
 * workspace: byte offsets from the workspace's start (the pointer passed as `workspace`), for a
 * workspace laid out for `shape` and `cfg`.  They let a caller (a test, a debugger, a profiler)
 * read the quantizer inputs, stage outputs and intermediate gradients of the last call, e.g. to
 * compare each stage of the block (Eq. 4 per linear, Eq. 5's attention, Eq. 1's loss) against
 * another implementation started from the same stage input.  The values stay valid until the
 * next call that uses the workspace.  Forward entries are written by both calls, backward
 * entries by omq_block_step only.  Per-token arrays [T] are one step h (fp32) and zero point z
 * (int32) per token row; qkv_h / qkv_z hold the q, k and v rows one after the other ([3, T]).
 * Weight entries are indexed 0 = q|k|v, 1 = o, 2 = gate|up, 3 = down: w_hat bf16 [Cout, Cin]
 * (the fake-quantized LET-scaled weight, Eq. 2 and Eq. 3), w_h fp32 and w_z int32
 * [Cout, ngroups]; w_hat[0] is -1 under cfg->wprep = 1 (the q|k|v W_hat is then never formed).
 * Returns OMQ_ERR_* for a shape or configuration omq_block_workspace_size rejects. */
typedef struct {
  int64_t a_hat;                   /* bf16 [T, d]: Q_a((RMSNorm(x) - d1) / s1), the q|k|v input */
  int64_t a_h, a_z;
  int64_t y_qkv;                   /* fp32 [T, nh*128 + 2*nkv*128]: q|k|v before RoPE (+ LET bias) */
  int64_t qkv_h, qkv_z;            /* of Q~, K~ (after RoPE and s_a) and V' */
  int64_t q_hat, k_hat, v_hat;     /* bf16 [T, nh*128], [T, nkv*128] x 2: Q_a(Q~), Q_a(K~), Q_a(V') */
  int64_t o;                       /* fp32 [T, nh*128]: attention output P V */
  int64_t o_hat, o_h, o_z;         /* bf16 [T, nh*128]: Q_a(O), the o_proj input */
  int64_t h1;                      /* fp32 [T, d]: x + o_proj output */
  int64_t b_hat, b_h, b_z;         /* bf16 [T, d]: Q_a((RMSNorm(h1) - d2) / s2) */
  int64_t y_gu;                    /* fp32 [T, 2 ffn]: gate | up (+ LET bias) */
  int64_t m_hat, m_h, m_z;         /* bf16 [T, ffn]: Q_a(silu(gate) up), the down_proj input */
  int64_t w_hat[4], w_h[4], w_z[4];
  int64_t dy;                      /* fp32 [T, d]: dL/dy */
  /* the intermediate gradients below are bf16, the operand of the products that take them (R13) */
  int64_t dy_gu;                   /* bf16 [T, 2 ffn]: dL/d(gate | up) */
  int64_t dh1;                     /* bf16 [T, d]: dL/dh1 (both paths) */
  int64_t do_bf16;                 /* bf16 [T, nh*128]: dL/dO through Q_a, the attention backward's operand */
  int64_t dy_qkv;                  /* bf16 [T, nh*128 + 2*nkv*128]: dL/d(q|k|v before RoPE) */
} omq_block_saved;
omq_status omq_block_saved_layout(const omq_block_shape* shape, const omq_qcfg* cfg, omq_block_saved* out);

/* Causal self-attention of the block (Sec. 3.3, Eq. 5 applies LET to Q and K before it; the
 * softmax output is not quantized), computed without storing the [T, T] scores.
 *   Q  [T, n_heads*128] bf16, row stride ldq; K, V [T, n_kv*128] bf16, row stride ldkv
 *      (query head h attends with kv head h / (n_heads / n_kv));
 *   O  [T, n_heads*128] fp32 out, row stride ldo: O = softmax(Q K^T / sqrt(128), causal) V;
 *   lse [n_heads, T] fp32 out: per row, log2 of sum_j exp2(c s_j - m) plus m, where
 *      c = log2(e)/sqrt(128) and s_j = q . k_j (the saved state the backward needs).
 * Head dimension 128 only (OMQ_ERR_SHAPE otherwise).  Strides in elements, multiples of 8 (bf16)
 * or 4 (fp32), base pointers 16-byte aligned (OMQ_ERR_ALIGN).  Device pointers, caller-owned;
 * enqueued on `stream`; a stalled pipeline writes OMQ_ERR_TIMEOUT to *dev_status (nullable). */
omq_status omq_attention_fwd(omq_stream_t stream, int32_t T, int32_t n_heads, int32_t n_kv, const void* Q,
                             int64_t ldq, const void* K, const void* V, int64_t ldkv, float* O, int64_t ldo,
                             float* lse, int32_t* dev_status);

/* Backward of omq_attention_fwd given dO [T, n_heads*128] bf16 (row stride lddo), the forward's
 * O and lse: dQ [T, n_heads*128] (row stride ldg), dK and dV [T, n_kv*128] (row stride ldgkv),
 * fp32, overwritten.  D [n_heads, T] fp32 is caller scratch (rowsum of dO * O).  The scores and
 * probabilities are recomputed from Q, K and lse. */
omq_status omq_attention_bwd(omq_stream_t stream, int32_t T, int32_t n_heads, int32_t n_kv, const void* Q,
                             int64_t ldq, const void* K, const void* V, int64_t ldkv, const float* O, int64_t ldo,
                             const float* lse, const void* dO, int64_t lddo, float* D, float* dQ, int64_t ldg,
                             float* dK, float* dV, int64_t ldgkv, int32_t* dev_status);

/* Softmax-output quantization variant of the attention (the ablation beside Table A7; off in the
 * method's default configuration).  As omq_attention_fwd, except that the probabilities of every
 * query row are fake-quantized with the MinMax quantizer of Eq. 2 (gamma = beta = 1, step floored at
 * h_eps) over the row's visible keys j <= t before the P V product; masked entries stay 0.
 *   pbits   2..8 (OMQ_ERR_UNSUPPORTED otherwise); h_eps > 0 (OMQ_ERR_INVALID_ARG otherwise);
 *   (a null pq_rows is OMQ_ERR_INVALID_ARG, a misaligned one OMQ_ERR_ALIGN)
 *   pq_rows [n_heads, T, 8] fp32 out, 16-byte aligned: per query row h, 1/h, z, the row's max and
 *           min probability, floored (0/1), the first key of the max and of the min (as exact
 *           floats). */
omq_status omq_attention_pq_fwd(omq_stream_t stream, int32_t T, int32_t n_heads, int32_t n_kv, const void* Q,
                                int64_t ldq, const void* K, const void* V, int64_t ldkv, float* O, int64_t ldo,
                                float* lse, int32_t pbits, float h_eps, float* pq_rows, int32_t* dev_status);

/* Backward of omq_attention_pq_fwd: straight-through estimator of the quantizer (R7 of the oracle:
 * the gradient passes inside the clamp range; h is not detached, the max and the min pass theirs to
 * their first key), then the softmax backward.  pq_rows is the forward's; pq_stats [n_heads, T, 4]
 * fp32 caller scratch, 16-byte aligned (per row sum_j P_j dP_j and the totals reaching the max and
 * the min).  Other arguments as omq_attention_bwd, without D. */
omq_status omq_attention_pq_bwd(omq_stream_t stream, int32_t T, int32_t n_heads, int32_t n_kv, const void* Q,
                                int64_t ldq, const void* K, const void* V, int64_t ldkv, const float* lse,
                                const void* dO, int64_t lddo, float* dQ, int64_t ldg, float* dK, float* dV,
                                int64_t ldgkv, int32_t pbits, const float* pq_rows, float* pq_stats,
                                int32_t* dev_status);

/* LET initialisation (Sec. 4.1 "Training": the channel-wise scaling is initialised as in
 * SmoothQuant, the channel-wise shifting as in Outlier Suppression+).  Column statistics of the
 * full-precision block over the calibration tokens, device fp32 vectors:
 *   a_*  [d]            ln1 output (the [ln1, (q,k,v)] pair's X)
 *   q_absmax [n_heads*hd], k_absmax [n_kv*hd]   Q and K after RoPE
 *   o_*  [n_heads*hd]   attention output (the [v, out] pair's X)
 *   b_*  [d]            ln2 output (the [ln2, (gate,up)] pair's X) */
typedef struct omq_let_stats {
  float* a_absmax; float* a_sum;
  float* q_absmax; float* k_absmax;
  float* o_absmax; float* o_sum;
  float* b_absmax; float* b_sum;
} omq_let_stats;

/* Runs the full-precision block (no quantization, no LET) on one calibration input x [T, d] fp32
 * and folds its column statistics into `stats` (first != 0 overwrites, else max / add).  The
 * workspace is the one omq_block_workspace_size gives for `shape` with wbits = abits = 16. */
omq_status omq_let_stats_accumulate(omq_stream_t stream, const omq_block_shape* shape,
                                    const omq_block_weights* w, const float* x, const omq_let_stats* stats,
                                    int32_t first, void* workspace, size_t ws_bytes, int32_t* dev_status);

size_t omq_let_init_workspace_size(const omq_block_shape* shape);

/* Initial LET parameters from the statistics of ntok calibration tokens, into theta's s1, d1,
 * so, do_, sa, s2, d2:  s = max(max|X|^alpha / max|W|^(1-alpha), 1e-5) per input channel with
 * max|W| over all output rows of the weights that share the input, delta = channel mean of X;
 * the [v, out] pair per value channel with maxima / means over the query heads of its group;
 * s_a = max(sqrt(max|Q| / max|K|), 1e-5), no Q/K shift.  alpha = 0.5 reproduces SmoothQuant's
 * default migration strength. */
omq_status omq_let_init(omq_stream_t stream, const omq_block_shape* shape, const omq_block_weights* w,
                        const omq_let_stats* stats, int64_t ntok, float alpha, const omq_block_params* theta,
                        void* workspace, size_t ws_bytes);

/* Fold & pack (Algorithm 1's last steps: transform the block with its learned parameters, then
 * quantize).  Per linear (q|k|v stacked, o, gate|up stacked, down): the integer codes of Eq. 2,
 * packed per output row as a little-endian bit stream (code i at bits [N i, N i + N), N = wbits,
 * Cin * N / 8 bytes per row), and h, z per group [Cout, Cin / group] (group 0: one per row).
 * With LET on, the LET parameters are absorbed: the linear biases B~ of Eq. 3 (the [v, out]
 * pair's shift and row scale inside q|k|v's v rows and o), the two RMSNorm layers as a gain 1/s and
 * a bias -delta/s (the block's RMSNorm has unit gain, no bias), and s_a, which scales Q and K after
 * RoPE and stays a runtime per-channel factor.  Device pointers, caller-owned; LET-only outputs
 * may be NULL when LET is off. */
typedef struct omq_block_packed {
  uint8_t* codes_qkv; uint8_t* codes_o; uint8_t* codes_gu; uint8_t* codes_d;
  float* h_qkv; int32_t* z_qkv; float* h_o; int32_t* z_o;
  float* h_gu; int32_t* z_gu; float* h_d; int32_t* z_d;
  float* b_qkv; float* b_o; float* b_gu;          /* [dq+2dkv], [d], [2 ffn] */
  float* ln1_gain; float* ln1_bias; float* ln2_gain; float* ln2_bias;   /* [d] */
  float* sa;                                      /* [n_kv*hd] */
} omq_block_packed;

size_t omq_block_pack_workspace_size(const omq_block_shape* shape, const omq_qcfg* cfg);
omq_status omq_block_fold_pack(omq_stream_t stream, const omq_block_shape* shape, const omq_block_weights* w,
                               const omq_block_params* theta, const omq_qcfg* cfg, const omq_block_packed* out,
                               void* workspace, size_t ws_bytes);

/* AdamW update of one fp32 parameter vector (Sec. 4.1 "Training": AdamW, weight decay 0):
 * m = b1 m + (1-b1) g; v = b2 v + (1-b2) g^2; p -= lr * (m / (1-b1^t)) / (sqrt(v / (1-b2^t)) + eps)
 * - lr * wd * p.  step t >= 1. */
omq_status omq_adamw_update(omq_stream_t stream, int64_t n, float* p, const float* g, float* m,
                            float* v, float lr, float beta1, float beta2, float eps,
                            float weight_decay, int32_t step);

/* The same update with the step count t read from device memory at *step_dev (int32, >= 1), so that
 * a captured CUDA graph replays correctly across steps.  Bias corrections 1 - b^t are formed on
 * the device in single precision. */
omq_status omq_adamw_update_dev(omq_stream_t stream, int64_t n, float* p, const float* g, float* m,
                                float* v, float lr, float beta1, float beta2, float eps,
                                float weight_decay, const int32_t* step_dev);

/* *step_dev += 1 on `stream` (one thread). */
omq_status omq_step_advance(omq_stream_t stream, int32_t* step_dev);

/* Reads the device status word written by kernels (synchronises `stream`).  *host_out receives
 * the word (0 = ok); the return value is OMQ_OK or OMQ_ERR_CUDA if the copy failed. */
omq_status omq_stream_status(omq_stream_t stream, const int32_t* dev_status, int32_t* host_out);

/* Human-readable name of a status code (static string). */
const char* omq_status_string(omq_status s);

/* Library version, for the bindings' sanity check. */
int32_t omq_version(void);

/* Number of kernel launches the library has enqueued since it was loaded (host-side counter). */
int64_t omq_launch_count(void);

/* Tracing of the tensor-core matrix products.  After omq_profile_begin, every omq GEMM launch is
 * bracketed by two CUDA events recorded on its own stream, and its algorithmic flop count (2 per
 * multiply-add inside the causal domain) is accumulated.  omq_profile_end waits for those events
 * and returns the summed device time in ms, the flops and the number of launches, then stops
 * tracing.  Not for use during CUDA-graph capture (it creates events lazily). */
void omq_profile_begin(void);
omq_status omq_profile_end(double* gemm_ms, double* gemm_flops, int64_t* gemm_launches);

#ifdef __cplusplus
}
#endif
#endif /* OMQ_H */
