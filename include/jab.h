/*
 * jab.h -- C ABI of the GB300 (sm_103a) library for the joint attention-block loss L_JAB.
 *
 * L_JAB (Section 2.2, Eq. 3, MSE term) compares the causal, GQA, RoPE attention output of one
 * transformer block computed with its float weights, A(X; W), against the same block computed with
 * the joint [W_Q | W_K | W_V] fake-quantised at b bits (Section 2.1, Eq. 2):
 *
 *     L_JAB(w_hat) = ||A(X; W) - A(X; w_hat)||_F^2 / (B * T * Hq * d_h)
 *
 * and its gradient w.r.t. the per-(row, group) scales uses the straight-through estimator on the
 * weights and the LSQ rule on the scales (App. B "Joint STE fine-tuning", Eq. 13).
 *
 * Conventions shared by every entry point
 *  - Pointers named *_dev are device pointers owned by the caller; the library never frees or
 *    retains them after the call is enqueued. Host arrays are named *_host.
 *  - Every entry point that takes a workspace uses only the caller's workspace `ws` (size from
 *    jab_workspace_size) for scratch. It allocates no device memory.
 *  - Calls are asynchronous on `stream`. Host-side argument checks return an error immediately and
 *    enqueue nothing. Problems found on the device (non-finite or non-positive scales, fp16 range
 *    overflow, a bounded wait that timed out) set a per-device flag that jab_get_device_status reads.
 *  - Layouts are row-major. The joint weight uses the nn.Linear layout: row o is output feature o,
 *    rows [0, Hq*d_h) are W_Q, then Hkv*d_h rows of W_K, then Hkv*d_h rows of W_V (a transpose would
 *    quantise along the wrong axis). Groups of G consecutive input columns share one scale.
 *  - bf16 and fp16 tensors are passed as `const void*` holding IEEE-754 binary16 / bfloat16 bits.
 *  - Supported shapes: head_dim in {64, 128}; d_model a multiple of 64; group_size a multiple of 64
 *    dividing d_model; n_q_heads a multiple of n_kv_heads; (Hq + 2 Hkv) * head_dim a multiple of 128;
 *    any B >= 1 and T >= 1 with B * T <= 2^31. Other shapes return JAB_ERR_UNSUPPORTED. Device
 *    pointers must be 16-byte aligned and the workspace 256-byte aligned.
 *  - The tensor-core operands of the forward path are fp16 (X and w_hat are converted from their
 *    bf16 inputs on the device); accumulation is fp32; the loss is summed in fp64.
 */
#ifndef JAB_H_
#define JAB_H_

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* Same handle type as cudaStream_t; NULL is the legacy default stream. */
typedef struct CUstream_st* jab_stream_t;

typedef enum {
  JAB_OK = 0,
  JAB_ERR_INVALID_ARG = 1,   /* NULL pointer, bad size, misaligned pointer, workspace too small   */
  JAB_ERR_UNSUPPORTED = 2,   /* shape outside the supported set above                            */
  JAB_ERR_CUDA = 3,          /* a CUDA runtime call or kernel launch failed                      */
  JAB_ERR_NONFINITE = 4,     /* device: scale <= 0 or non-finite, or a non-finite result          */
  JAB_ERR_RANGE = 5,         /* device: a value does not fit the fp16 tensor-core operands: X, the
                                quantised weights, the projected Q|K|V or the output error dO
                                (|x| > 65504 after rounding)                                    */
  JAB_ERR_TIMEOUT = 6,       /* device: a bounded wait in a pipelined kernel gave up             */
  JAB_ERR_SCRATCH_LIMIT = 7, /* jab_loss_forward_noalloc: the problem needs more scratch than the
                                fixed JAB_NOALLOC_SCRATCH_BYTES                                    */
  JAB_ERR_INTERNAL = 8,      /* device: an internal invariant did not hold (e.g. the alignment of
                                a kernel's shared memory); the kernel returned without work     */
  JAB_ERR_DEVICE_ASSERT = 9  /* device, checked build only (libjab_checked.so): an index was
                                outside its buffer; the access was skipped                       */
} jab_status;

/* One attention block. Section 2.1 (d, d_head), App. C (Mistral-7B: GQA, RoPE theta = 1e4). */
typedef struct {
  int32_t d_model;      /* d: input features of X and columns of W                               */
  int32_t n_q_heads;    /* Hq                                                                     */
  int32_t n_kv_heads;   /* Hkv; query head h reads key/value head h / (Hq / Hkv)                  */
  int32_t head_dim;     /* d_h                                                                    */
  int32_t group_size;   /* G: input columns per scale                                             */
  int32_t use_rope;     /* 0: no RoPE (GPT-2); 1: rotate-half RoPE on Q and K, positions 0..T-1    */
  float rope_theta;     /* RoPE base; inv_freq_j = theta^(-2j/d_h)                                 */
  float softmax_scale;  /* <= 0 selects 1/sqrt(d_h) (Section 2.1)                                  */
} jab_block_desc;

/* Bytes of workspace the calls below need for this block, B sequences of T tokens, n_cand candidates
 * per jab_loss_forward call, with_bwd != 0 for jab_loss_backward_scales. Returns 0 on invalid input.
 * One workspace sized with (n_cand = max, with_bwd = 1) serves every entry point. */
size_t jab_workspace_size(const jab_block_desc* desc, int32_t B, int32_t T, int32_t n_cand,
                          int32_t with_bwd);

/* Teacher pass (Section 2.2: A(X) of the unmodified block; App. B, decision 3: teacher and student
 * see the same X). Computes A(X; W) once per block; its cost is shared by every candidate.
 *   X_dev          bf16 [B, T, d_model]
 *   W_dev          bf16 [(Hq + 2 Hkv) * d_h, d_model]   (nn.Linear layout, see above)
 *   A_ref_dev      out fp32 [B, T, Hq * d_h]            merged heads, pre-o_proj
 *   lse_dev        out fp32 [B, Hq, T] or NULL          log-sum-exp of each softmax row
 *   a_sqnorm_dev   out fp64 [1] or NULL                 ||A_ref||_F^2 (for eps^A = sqrt(SSE/||A||^2)) */
jab_status jab_reference_forward(const jab_block_desc* desc, int32_t B, int32_t T,
                                 const void* X_dev, const void* W_dev, float* A_ref_dev,
                                 float* lse_dev, double* a_sqnorm_dev, void* ws, size_t ws_bytes,
                                 jab_stream_t stream);

/* Forward L_JAB (Eq. 3, MSE term) for n_cand candidate (bits, scales) pairs of the same block, e.g.
 * the bit widths scored for the knapsack (Section 2.4). X is read once for all candidates.
 *   bits_host      int32 [n_cand], each in [2, 8]
 *   scales_host    host array [n_cand] of device pointers, each fp32 [(Hq+2Hkv)*d_h, d_model/G] > 0
 *   loss_dev       out fp64 [n_cand]                    SSE_c / (B * T * Hq * d_h)
 *   sse_parts_dev  out fp64 [n_cand, B, Hq] or NULL     SSE of each (candidate, sequence, query head) */
jab_status jab_loss_forward(const jab_block_desc* desc, int32_t B, int32_t T, const void* X_dev,
                            const void* W_dev, const float* A_ref_dev, int32_t n_cand,
                            const int32_t* bits_host, const float* const* scales_host,
                            double* loss_dev, double* sse_parts_dev, void* ws, size_t ws_bytes,
                            jab_stream_t stream);

/* Teacher projection for the KL term of Eq. 3: the rotated [Q | K | V] = RoPE(X W^T) of the block
 * with its float weights, in fp16 (the operand type of the tensor-core path), computed once per
 * block like A_ref. Only its Q and K columns are read by jab_loss_forward_kl.
 *   QKV_ref_dev    out fp16 [B, T, (Hq + 2 Hkv) * d_h], 16-byte aligned
 *   ws             at least jab_workspace_size(desc, B, T, 1, 0) bytes
 * A projected value outside the fp16 range raises JAB_ERR_RANGE on the device. */
jab_status jab_reference_projection(const jab_block_desc* desc, int32_t B, int32_t T,
                                    const void* X_dev, const void* W_dev, void* QKV_ref_dev,
                                    void* ws, size_t ws_bytes, jab_stream_t stream);

/* Forward L_JAB with both terms of Eq. 3 for n_cand candidates: the MSE term of jab_loss_forward
 * plus lambda_kl times the KL attention-map term D_KL(P || Q) between the teacher's post-softmax
 * map P and each candidate's map Q, with the batchmean normalisation the paper implements (App. B
 * "Effective weight of the KL term"): the sum over sequences, query heads, query rows and visible
 * keys of P log(P / Q), divided by B. The paper's default is lambda_kl = 0.1 (Section 3).
 *   QKV_ref_dev    fp16 [B, T, D] from jab_reference_projection for the same X and W
 *   lambda_kl      >= 0
 *   loss_dev       out fp64 [n_cand]   mse + lambda_kl * kl
 *   mse_dev        out fp64 [n_cand] or NULL   the MSE term (as jab_loss_forward's loss)
 *   kl_dev         out fp64 [n_cand] or NULL   the KL term
 *   kl_rows_dev    out fp32 [n_cand, B, Hq, T] or NULL   KL of every query row (nats)
 * Other arguments as for jab_loss_forward; ws of jab_workspace_size(desc, B, T, n_cand, 0). */
jab_status jab_loss_forward_kl(const jab_block_desc* desc, int32_t B, int32_t T, const void* X_dev,
                               const void* W_dev, const float* A_ref_dev, const void* QKV_ref_dev,
                               int32_t n_cand, const int32_t* bits_host,
                               const float* const* scales_host, float lambda_kl, double* loss_dev,
                               double* mse_dev, double* kl_dev, float* kl_rows_dev, void* ws,
                               size_t ws_bytes, jab_stream_t stream);

/* Hutchinson estimate of Tr(H), the trace of the Hessian of L_JAB (MSE term) w.r.t. the joint
 * weights at the float point (Section 2.4, Eq. 5): Tr(H) ~ (1/m) sum_i v_i^T H v_i over m
 * Rademacher probes v_i. At the float weights H = 2 J_A^T J_A / n (n = B T Hq d_h), so each probe
 * costs one forward-mode (JVP) pass: v^T H v = 2 ||J_A v||^2 / n, with J_A v the derivative of the
 * block output along v (the tangent projection X v^T through the same RoPE, then the attention
 * JVP), no second backward pass.
 * Probe i, entry e (row-major over [(Hq+2Hkv) d_h, d_model]) is -1 when the top bit of the
 * (i * (Hq+2Hkv) d_h d_model + e + 1)-th output of SplitMix64 (Steele, Lea and Flood, 2014)
 * seeded with `seed` is set, else +1. The probe enters the tensor-core path scaled by the exact
 * power of two 2^-k, k = floor(log2(sqrt(d_model))), so that the tangent projections stay in the
 * fp16 range; the quadratic form is rescaled by 4^k (exactly). A tangent value that still leaves
 * the fp16 range raises JAB_ERR_RANGE on the device.
 *   A_ref_dev, lse_ref_dev  the teacher pass of jab_reference_forward (lse_ref required)
 *   trace_dev      out fp64 [1]            the estimate
 *   vhv_dev        out fp64 [n_probes] or NULL   v_i^T H v_i of each probe
 *   ws             at least jab_workspace_size(desc, B, T, 2, 0) bytes */
jab_status jab_hutchinson_trace(const jab_block_desc* desc, int32_t B, int32_t T,
                                const void* X_dev, const void* W_dev, const float* A_ref_dev,
                                const float* lse_ref_dev, int32_t n_probes, uint64_t seed,
                                double* trace_dev, double* vhv_dev, void* ws, size_t ws_bytes,
                                jab_stream_t stream);

/* The probe entries of jab_hutchinson_trace: entries first .. first + n - 1 of the probe sequence
 * of `seed` (probe i, entry e is number i * (Hq+2Hkv) d_h d_model + e) as fp16 -1 / +1.
 *   out_dev        out fp16 [n], 16-byte aligned; n a multiple of 8 */
jab_status jab_rademacher_probes(uint64_t seed, int64_t first, int64_t n, void* out_dev,
                                 jab_stream_t stream);

/* Sensitivity scores of Eq. 6 for n_cand candidate (bits, scales) quantisations of the block:
 *   C1: Omega(b) = Tr(H) ||Q_b(W) - W||_F^2,   C2: (L - i) Omega(b) with layers_after = L - i.
 *   trace_dev      fp64 [1] on the device (e.g. from jab_hutchinson_trace)
 *   c1_dev         out fp64 [n_cand];  c2_dev  out fp64 [n_cand] or NULL
 *   ws             at least jab_workspace_size(desc, 1, 1, n_cand, 0) bytes
 * The squared error is summed in fp64 in a fixed order (repeated calls give identical bits). */
jab_status jab_omega_scores(const jab_block_desc* desc, const void* W_dev, int32_t n_cand,
                            const int32_t* bits_host, const float* const* scales_host,
                            const double* trace_dev, int32_t layers_after, double* c1_dev,
                            double* c2_dev, void* ws, size_t ws_bytes, jab_stream_t stream);

/* Forward L_JAB and its gradient w.r.t. the scales for one candidate (App. B "Joint STE fine-tuning",
 * Eq. 13): d w_hat / d w = 1 (STE) and d w_hat / d s = q - v if |v| <= qmax, else sign(v) qmax, with
 * v = w / s.
 *   grad_scales_dev out fp32 [(Hq+2Hkv)*d_h, d_model/G] = kappa * sum_{i in group} dL/dw_hat[o,i] * r[o,i]
 *   kappa          <= 0 selects the LSQ factor (G * qmax)^(-1/2); 1 gives the raw rule
 *   loss_dev       out fp64 [1]
 * The gradient's sums (over tokens in the GEMM, then over the GEMM's K splits) run in a fixed order:
 * repeated calls with identical inputs return identical bits. */
jab_status jab_loss_backward_scales(const jab_block_desc* desc, int32_t B, int32_t T,
                                    const void* X_dev, const void* W_dev, const float* A_ref_dev,
                                    int32_t bits, const float* scales_dev, float kappa,
                                    double* loss_dev, float* grad_scales_dev, void* ws,
                                    size_t ws_bytes, jab_stream_t stream);

/* The STE fitting loop (App. B "Joint STE fine-tuning": 200 steps per block on one fixed calibration
 * batch) evaluates the same X at every step. jab_prepare_x converts X once into the fp16 copy that
 * the projection reads, kept in `ws`; jab_loss_backward_scales_prepared is then
 * jab_loss_backward_scales without that conversion. Its arguments and results are those of
 * jab_loss_backward_scales; X_dev must be the same pointer (with the same contents, B and T) as in
 * the last call that converted X into this workspace (jab_prepare_x or any entry point taking X),
 * otherwise it returns JAB_ERR_INVALID_ARG. X_dev is still read (in bf16) by the weight-gradient
 * GEMM. jab_prepare_x: ws of at least jab_workspace_size(desc, B, T, 1, 0) bytes; X out of the
 * fp16 range raises JAB_ERR_RANGE on the device. */
jab_status jab_prepare_x(const jab_block_desc* desc, int32_t B, int32_t T, const void* X_dev,
                         void* ws, size_t ws_bytes, jab_stream_t stream);
jab_status jab_loss_backward_scales_prepared(const jab_block_desc* desc, int32_t B, int32_t T,
                                             const void* X_dev, const void* W_dev,
                                             const float* A_ref_dev, int32_t bits,
                                             const float* scales_dev, float kappa,
                                             double* loss_dev, float* grad_scales_dev, void* ws,
                                             size_t ws_bytes, jab_stream_t stream);

/* The STE / LSQ scale gradient of the joint objective of Eq. 3, L = MSE + lambda_kl * KL, with the
 * KL term D_KL(P || Q) between the teacher's attention map P and the student's Q in the batchmean
 * normalisation (App. B "Effective weight of the KL term"; the paper's default lambda_kl = 0.1,
 * Section 3). The KL term adds (lambda_kl / B)(Q - P) to the gradient with respect to the student's
 * scaled scores (P, Q: post-softmax maps), which then flows through the same dQ / dK products,
 * the transpose of RoPE, the weight-gradient GEMM and the LSQ rule (Eq. 13) as the MSE term's.
 *   QKV_ref_dev    fp16 [B, T, (Hq + 2 Hkv) * d_h] from jab_reference_projection (same X and W),
 *                  16-byte aligned
 *   lse_ref_dev    fp32 [B, Hq, T]: the teacher's row log-sum-exp from jab_reference_forward
 *                  (natural log, scaled scores)
 *   lambda_kl      >= 0 (0 gives jab_loss_backward_scales' gradient through the KL code path)
 *   loss_dev       out fp64 [1]   MSE + lambda_kl * KL
 *   kl_dev         out fp64 [1] or NULL   the KL term (nats, batchmean)
 * Other arguments, layouts and errors as for jab_loss_backward_scales (X is converted by the call);
 * ws of jab_workspace_size(desc, B, T, 1, 1) bytes. The score gradient is held in fp16 tiles as
 * a P (dP - D) + b (P - P_teacher) with b / a = lambda_kl B T Hq d_h / (2 B) and b <= 1024, so
 * where the KL term dominates, the MSE term's share below the fp16 resolution of the sum is lost. */
jab_status jab_loss_backward_scales_kl(const jab_block_desc* desc, int32_t B, int32_t T,
                                       const void* X_dev, const void* W_dev,
                                       const float* A_ref_dev, const void* QKV_ref_dev,
                                       const float* lse_ref_dev, int32_t bits,
                                       const float* scales_dev, float kappa, float lambda_kl,
                                       double* loss_dev, double* kl_dev, float* grad_scales_dev,
                                       void* ws, size_t ws_bytes, jab_stream_t stream);

/* Forward L_JAB and the STE weight gradient for one candidate (App. B "Joint STE fine-tuning":
 * d w_hat / d w = 1, so dL/dW = dL/dw_hat), and its squared Frobenius norm: the Fisher-coupling score
 * of App. B "Fisher-coupling" when called with bits = 2 and round-to-nearest scales
 * (jab_init_scales mode 0).
 *   grad_w_dev      out fp32 [(Hq+2Hkv)*d_h, d_model] or NULL   dL/dw_hat = (2/n) dQKV^T X, n = B*T*Hq*d_h
 *   grad_sqnorm_dev out fp64 [1] or NULL                        ||dL/dw_hat||_F^2, reduced from the
 *                                                               stored gradient in a fixed order
 * The weight-gradient GEMM may split the token range and add the partial tiles with atomics, so the
 * last bits of grad_w (and of its norm) may differ between calls; in the deterministic-reduction
 * mode (jab_set_deterministic) each tile is one unit and repeated calls are bit-identical.
 *   loss_dev        out fp64 [1]
 * At least one of grad_w_dev and grad_sqnorm_dev must be non-NULL. Uses the with_bwd workspace of
 * jab_workspace_size. */
jab_status jab_loss_backward_weights(const jab_block_desc* desc, int32_t B, int32_t T,
                                     const void* X_dev, const void* W_dev, const float* A_ref_dev,
                                     int32_t bits, const float* scales_dev, double* loss_dev,
                                     float* grad_w_dev, double* grad_sqnorm_dev, void* ws,
                                     size_t ws_bytes, jab_stream_t stream);

/* Bit-width allocation over L layers (Section 2.4, Eq. 7; App. B "Allocators"). Host code only: no
 * device memory, no CUDA call, synchronous.
 * Minimises sum_i omega[i, b_i] subject to sum_i n_i b_i <= avg_bits * sum_i n_i (the parameter-
 * weighted budget of Eq. 8: c(b_i) = n_i b_i).
 * The walk (App. B "Allocators"):
 *   - every layer starts at its highest width;
 *   - while over budget, apply the one-step downgrade with the least score increase per bit saved;
 *   - then, while one fits and lowers the total, apply the one-step upgrade with the largest score
 *     decrease per bit.
 * Ties go to the lowest layer index.
 *   omega_host      fp64 [L, n_widths]  finite score of layer i at widths_host[k]: direct L_JAB
 *                                       (jab_loss_forward), or Omega C1 / C2 of Eq. 6
 *   widths_host     int32 [n_widths]    strictly increasing bit widths, e.g. {2, 3, 4, 8, 16}
 *   n_weights_host  int64 [L]           weights of each layer: a layer at width b costs n_i * b bits
 *   avg_bits        average bits per weight allowed
 *   method          0: walk over every width (greedy); 1: walk over each layer's Pareto-efficient
 *                   points only (a point is dropped when a cheaper one scores no worse)
 *   bits_out_host   out int32 [L]
 * Returns JAB_ERR_INVALID_ARG for NULL pointers, sizes < 1, non-increasing widths, non-finite
 * scores, or a budget below the cost of every layer at its lowest width. */
jab_status jab_allocate_bits(const double* omega_host, const int32_t* widths_host,
                             const int64_t* n_weights_host, int32_t L, int32_t n_widths,
                             double avg_bits, int32_t method, int32_t* bits_out_host);

/* Quantiser alone (Section 2.1, Eq. 2): v = fl32(w / s), q = clip(round-half-even(v), -qmax, qmax).
 *   codes_dev      out int8 [(Hq+2Hkv)*d_h, d_model] or NULL
 *   w_hat_dev      out fp32 [(Hq+2Hkv)*d_h, d_model] or NULL   fl32(q * s) */
jab_status jab_quantize(const jab_block_desc* desc, int32_t bits, const void* W_dev,
                        const float* scales_dev, int8_t* codes_dev, float* w_hat_dev,
                        jab_stream_t stream);

/* Flip count (App. B "Joint STE fine-tuning", Eq. 15): the number of grid positions whose code
 * differs between two code arrays of the same weights, e.g. after and before fine-tuning (codes
 * from jab_quantize). The flip rate is *count_dev / n.
 *   codes_a_dev, codes_b_dev  int8 [n], 16-byte aligned (may be NULL when n = 0)
 *   count_dev                 out int64 [1], 8-byte aligned (exact integer count; the same on
 *                             every call) */
jab_status jab_flip_rate(const int8_t* codes_a_dev, const int8_t* codes_b_dev, int64_t n,
                         int64_t* count_dev, jab_stream_t stream);

/* Starting scales. mode 0: max_{i in g}|w| / qmax (an all-zero group gets 1). mode 1: the per-group
 * min-MSE search over s_k = fl32(s_0 * (100 - k) / 100), k = 0..79, minimising
 * sum_{i in g} (Q(w_i; s_k) - w_i)^2 (ties to the smallest k).
 *   scales_dev     out fp32 [(Hq+2Hkv)*d_h, d_model/G] */
jab_status jab_init_scales(const jab_block_desc* desc, int32_t bits, int32_t mode,
                           const void* W_dev, float* scales_dev, jab_stream_t stream);

/* Bytes of the fixed device scratch array behind jab_loss_forward_noalloc (64 MiB). */
#define JAB_NOALLOC_SCRATCH_BYTES ((size_t)64 << 20)

/* jab_loss_forward without a caller workspace, for callers that cannot allocate device memory (all
 * of it reserved up front by another allocator, or allocation forbidden where the loss is needed).
 * The paper has no counterpart: this is a deployment convenience around the same computation.
 * Arguments and results are those of jab_loss_forward minus ws / ws_bytes; the scratch is one
 * file-scope device array of JAB_NOALLOC_SCRATCH_BYTES that every GPU loading this library holds
 * until the process exits. Problems whose jab_workspace_size(desc, B, T, n_cand, 0) exceeds it
 * return JAB_ERR_SCRATCH_LIMIT (e.g. a GPT-2-sized block with a few candidates and a few thousand
 * tokens fits; a full Mistral-sized calibration batch does not). The first call on a device looks
 * up the array's device address (cudaGetSymbolAddress), so make that first call before any stream
 * capture. No memory is allocated or freed by any call. All calls share the one array: calls that
 * overlap on the GPU (different streams, no ordering between them) race on it; serialise them. */
jab_status jab_loss_forward_noalloc(const jab_block_desc* desc, int32_t B, int32_t T,
                                   const void* X_dev, const void* W_dev, const float* A_ref_dev,
                                   int32_t n_cand, const int32_t* bits_host,
                                   const float* const* scales_host, double* loss_dev,
                                   double* sse_parts_dev, jab_stream_t stream);

/* Failure-path self-test (not part of the method): launches one CTA that waits, with the bounded
 * mbarrier wait of every pipelined kernel, on a barrier phase nothing completes. After the wait's
 * 2-second limit the kernel sets JAB_ERR_TIMEOUT in the device status and returns; the context
 * stays usable. Read the result with jab_get_device_status. */
jab_status jab_selftest_wait_timeout(jab_stream_t stream);

/* Deterministic-reduction mode (the boundary's "bit-identical results" convention), process-wide,
 * read when a call is issued: on = 1 makes every floating-point reduction of the library run in a
 * fixed order, so that two calls with identical inputs return bit-identical results; on = 0 (the
 * default) lets the weight-gradient GEMM of jab_loss_backward_weights split the token range and add
 * its partial tiles with atomics (faster on large batches; the last bits of grad_w may then differ).
 * Every other result (losses, scale gradients, KL, Hutchinson and Omega sums, norms) is reduced in a
 * fixed order in both modes. Returns JAB_ERR_INVALID_ARG for other values of on. Host only. */
jab_status jab_set_deterministic(int32_t on);

/* Self-test of the checked build's bounds checks: a one-block kernel writes buf_dev[i] = i for
 * i = 0 .. n, one index past the n-element extent it is given, each write behind the check. In the
 * checked build the last write is skipped and the device status becomes JAB_ERR_DEVICE_ASSERT
 * (buf_dev[n] keeps its value: give the buffer n + 1 elements to see it). The normal build launches
 * nothing and returns JAB_ERR_UNSUPPORTED. JAB_ERR_INVALID_ARG for a NULL buffer or n < 1. */
jab_status jab_selftest_bounds_check(int32_t* buf_dev, int32_t n, jab_stream_t stream);

/* Synchronises `stream`, then returns and clears the device-side status of the current device
 * (JAB_OK if no kernel reported a problem since the last call). */
jab_status jab_get_device_status(jab_stream_t stream);

/* ---- Instrumentation (not part of the method): per-launch-site device time with CUDA events. ----
 * jab_timing_enable(1) makes every later entry-point call record a CUDA event pair on its stream
 * around each of its kernel launch sites. jab_timing_collect synchronises those events and folds
 * them into per-site totals; jab_timing_get(i, ...) reads site i (0 <= i < jab_timing_count()):
 * its name, the summed device time in ms, the number of recorded ranges and the number of kernels
 * launched. jab_timing_reset clears the totals. Host-side state, guarded by a mutex. */
jab_status jab_timing_enable(int32_t on);
jab_status jab_timing_collect(void);
int32_t jab_timing_count(void);
jab_status jab_timing_get(int32_t i, const char** name, double* total_ms, int64_t* ranges,
                          int64_t* kernels);
jab_status jab_timing_reset(void);

/* Static, NUL-terminated description of a status code. */
const char* jab_status_string(jab_status status);

#ifdef __cplusplus
}
#endif

#endif /* JAB_H_ */
