/*
 * p4q.h - C ABI of the P4Q pruned W4A4 hot path on NVIDIA GB300 (sm_103a).
 *
 * P4Q (co-designed visual-token pruning and W4A4 quantization) runs two things
 * between the vision projector and the low-bit language model:
 *   1. a quantization-aware visual-token selector (Sec. 3.2, Eq. 4): the
 *      projector features and the question's concept embeddings are copied,
 *      fake-quantized to 4 bits, and scored in three sequential stages (query
 *      relevance per concept, CLS saliency, greedy max-min diversity) until the
 *      token budget K is filled; the original FP16 features of the kept tokens
 *      are forwarded;
 *   2. W4A4 linear layers on the shortened sequence (App. A and App. B.3):
 *      symmetric round-to-nearest INT4 weights with one scale per output
 *      channel, INT4 activations with one scale per token, integer matmul and
 *      dequantization.
 *
 * Conventions shared by every entry point
 *   - Pointers are DEVICE pointers unless a parameter says otherwise. The
 *     caller owns every buffer; the library allocates nothing per call.
 *   - fp16 tensors are passed as uint16_t bit patterns (IEEE binary16).
 *   - Packed INT4: two codes per byte, the even index in the low nibble, each
 *     nibble a two's complement integer. Codes produced here lie in [-7, 7].
 *   - All work is enqueued asynchronously on `stream` (NULL = legacy default
 *     stream); p4q_stream_t has the same type as cudaStream_t.
 *   - Arguments are validated on the host before anything is launched; a
 *     failed check returns an error status and launches nothing.
 *     P4Q_ERR_CUDA reports a launch error (query cudaGetLastError for detail).
 *     Device-side waits are bounded: a wait that runs out sets a device error
 *     word, the kernel returns, and the next p4q_device_status() call reports
 *     P4Q_ERR_TIMEOUT. No call aborts the process or traps the GPU.
 *   - Behaviour on non-finite inputs is unspecified (no fault, values undefined).
 *   - Alignment: every device pointer must be 16-byte aligned.
 */
#ifndef P4Q_H_
#define P4Q_H_

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef struct CUstream_st* p4q_stream_t;

typedef enum {
  P4Q_OK = 0,
  P4Q_ERR_INVALID_ARG = 1,          /* null pointer, negative size, K > N, ... */
  P4Q_ERR_UNSUPPORTED_SHAPE = 2,    /* size outside the documented limits */
  P4Q_ERR_MISALIGNED = 3,           /* a device pointer not 16-byte aligned */
  P4Q_ERR_WORKSPACE_TOO_SMALL = 4,  /* ws_bytes below the queried size */
  P4Q_ERR_CUDA = 5,                 /* a CUDA runtime / launch error */
  P4Q_ERR_TIMEOUT = 6,              /* a bounded device wait ran out */
  P4Q_ERR_NO_DEVICE = 7             /* no sm_103 device current */
} p4q_status;

/* Budget split of the selector (Sec. 3.2: alpha = 0.3, beta = 0.2, gamma =
 * 0.5). K_q = floor(alpha_permille * K / 1000) tokens go to query relevance,
 * K_s = floor(beta_permille * K / 1000) to CLS saliency, the rest
 * K_d = K - K_q - K_s to diversity. When no concept embeddings are given
 * (Q == NULL or J == 0) K_q moves to diversity; when A_cls == NULL K_s does. */
typedef struct {
  int32_t K;               /* retained visual tokens per image, 1 <= K <= N */
  int32_t alpha_permille;  /* query-relevance share, 0..1000 (default 300) */
  int32_t beta_permille;   /* saliency share, 0..1000-alpha (default 200) */
} p4q_select_params;

/* Limits checked by the calls below. */
#define P4Q_MAX_TOKENS 4096   /* N, visual tokens per image */
#define P4Q_MAX_CONCEPTS 16   /* J, concept embeddings per image */
#define P4Q_MAX_ROW 16384     /* d and Kin (elements per row) */

/* Human-readable name of a status code (static storage, never NULL). */
const char* p4q_status_string(p4q_status s);

/* Reads and clears the device error word of the current device after
 * synchronizing `stream`. Returns P4Q_ERR_TIMEOUT if a bounded device wait ran
 * out since the last call, P4Q_ERR_CUDA on a CUDA error, else P4Q_OK. */
p4q_status p4q_device_status(p4q_stream_t stream);

/* Number of kernels this library has launched in the process so far (all
 * devices, all streams). Host-side counter for launch accounting; no device
 * work. */
uint64_t p4q_launch_count(void);

/* GEMM kernel variant used by p4q_w4a4_linear and p4q_w4a4_gemm_s32, for all
 * later calls in the process (for tests and tuning; results are identical):
 *   0 automatic (default): for M <= 8 rows a weight-streaming kernel (dp4a
 *     on the CUDA cores: the packed weights are read once); CTA-pair kernel
 *     for fp16 outputs with M >= 256 and N >= 256; single-CTA kernel
 *     otherwise;
 *   1 single-CTA kernel only;
 *   2 CTA-pair kernel whenever N >= 256 (also for int32 outputs);
 *   3 like 0, and the workspace entry points take the expanded-operand path
 *     whenever a workspace is given (also below M = 512).
 * Variants 1 and 2 also keep the workspace entry points on the in-kernel
 * unpack. Returns P4Q_ERR_INVALID_ARG for other values. Not thread-safe
 * against concurrent launches. */
p4q_status p4q_set_gemm_variant(int variant);

/* Test of the bounded-wait path: launches one warp that waits on an mbarrier
 * nothing ever completes. The wait gives up after limit_us microseconds, sets
 * the device error word exactly as a stalled GEMM pipeline would, and the
 * kernel returns; the next p4q_device_status() on the same stream reports
 * P4Q_ERR_TIMEOUT (and clears it), and the context stays usable. The paper
 * has no counterpart: this exists so that failure detection is testable
 * without a GPU fault.
 *   limit_us  1 .. 1000000 (else P4Q_ERR_INVALID_ARG; nothing is launched)
 * Asynchronous on `stream`. */
p4q_status p4q_test_wait_timeout(uint32_t limit_us, p4q_stream_t stream);

/* Throughput probe for the roofline denominators of the integer
 * contractions. The paper has no counterpart: the W4A4 GEMM runs its exact
 * integer products on the FP8 tensor pipe (sm_103a has no integer tcgen05
 * MMA kind), and these loops measure what each candidate pipe sustains on
 * this GPU, with operands that stay on chip:
 *   kind 0  tcgen05.mma kind::f8f6f4 (E4M3 x E4M3 -> F32, M 256 x N 256 x
 *           K 32 per instruction, one CTA pair per two SMs), iters x 4 MMAs
 *           per pair;
 *   kind 1  mma.sync m16n8k32 s8 x s8 -> s32, 8 independent accumulators per
 *           warp, 32 warps per SM, iters rounds;
 *   kind 2  dp4a (s8 x 4 -> s32), 8 chains per thread, iters rounds.
 *   iters   1 .. 2^24
 *   sink    device buffer of at least 8192 uint32 (written only by a result
 *           that never occurs in practice; it keeps the work live)
 *   ops     HOST pointer: receives the number of operations the launch
 *           performs (2 per multiply-add)
 * Time the call with CUDA events on `stream`; ops / time is the rate.
 * Asynchronous; P4Q_ERR_INVALID_ARG for other kinds or iters. */
p4q_status p4q_peak_probe(int kind, int iters, uint32_t* sink, double* ops, p4q_stream_t stream);

/* ---------------------------------------------------------------------- */
/* Per-row 4-bit quantizers (App. A, App. B.3)                             */
/* ---------------------------------------------------------------------- */

/* Per-token activation quantization (App. A: symmetric round-to-nearest,
 * per-token 4-bit activations, group size -1, clip ratio 1.0).
 * For each row m of X:
 *   a = max_k |X[m,k]|, s_a[m] = a / 7 (fp32, rounded once),
 *   code[m,k] = clamp(round_half_even(X[m,k] / s_a[m]), -8, 7) with the
 *   quotient rounded to fp32; a == 0 gives s_a[m] = 0 and zero codes.
 *   X   [M, Kin] fp16 row-major (device, read)
 *   Xq  [M, Kin/2] packed INT4 (device, written)
 *   s_a [M] fp32 (device, written)
 * Requires M >= 0, 2 <= Kin <= P4Q_MAX_ROW, Kin % 16 == 0. M == 0 is a no-op. */
p4q_status p4q_quant_act(const uint16_t* X, int M, int Kin, uint8_t* Xq, float* s_a,
                         p4q_stream_t stream);

/* p4q_quant_act on rows that lie ldx elements apart: row m of X starts at
 * X + m * ldx (a column block of a wider matrix, e.g. the q part of a fused
 * q/k/v output). Same computation and outputs (Xq and s_a stay dense).
 * Requires ldx >= Kin and ldx % 8 == 0 (16-byte aligned rows); otherwise as
 * p4q_quant_act. */
p4q_status p4q_quant_act_ld(const uint16_t* X, int ldx, int M, int Kin, uint8_t* Xq, float* s_a,
                            p4q_stream_t stream);

/* p4q_quant_act_ld that also writes the codes in the expanded form of
 * p4q_expand_codes (Xu [M, Kin] bytes, sum_xu [M] int32), for
 * p4q_w4a4_linear_expanded, without a second pass. The paper has no
 * counterpart. */
p4q_status p4q_quant_act_expanded(const uint16_t* X, int ldx, int M, int Kin, uint8_t* Xq, float* s_a, uint8_t* Xu,
                                  int32_t* sum_xu, p4q_stream_t stream);

/* SwiGLU before down_proj fused with the per-token quantizer of its input
 * (App. A quantizes every linear's input per token; the decoder's MLP feeds
 * down_proj with silu(gate) * up). For each row m:
 *   h_k = silu(g_k) * u_k, silu(g) = g / (1 + e^-g), evaluated in fp32 as
 *   g * (1 / (1 + exp32(-g))) (each operation one rounded fp32 step, the
 *   reciprocal correctly rounded), where exp32 is this library's own fp32
 *   exponential (Cody-Waite reduction with ln2 = 355/512 + a low part, the
 *   degree-7 Taylor polynomial, two exact power-of-two scalings: within
 *   0.9 ulp of e^x; 0 for x < -87, inf for x > 88.72284, so silu(g) = 0
 *   for g < -88.72284);
 *   then the codes and scale of h as p4q_quant_act. h is within 2.9 ulp
 *   (3.5e-7 relative) of the real silu(g) * u, so the scale is within 1e-6
 *   of the exact one, the quotient h / s within 5.7e-6 of the exact
 *   quotient, and every code equals the code of the exact h except where
 *   that quotient lies within 5.7e-6 of a .5 boundary.
 *   gate, up [M, Kin] fp16, rows ld_gate / ld_up elements apart (column
 *              blocks of a fused gate|up output; device, read)
 *   Xq [M, Kin/2], s_a [M]           written
 *   Xu [M, Kin], sum_xu [M]          the expanded codes (p4q_expand_codes
 *                                    form) or both NULL
 * Requires M >= 0, 16 <= Kin <= P4Q_MAX_ROW, Kin % 16 == 0, ld >= Kin,
 * ld % 8 == 0, 16-byte aligned pointers. M == 0 is a no-op. */
p4q_status p4q_swiglu_quant_expanded(const uint16_t* gate, int ld_gate, const uint16_t* up, int ld_up, int M, int Kin,
                                     uint8_t* Xq, float* s_a, uint8_t* Xu, int32_t* sum_xu, p4q_stream_t stream);

/* RMSNorm before the quantized linears fused with the per-token quantizer of
 * its output (App. A quantizes every linear's input per token; the decoder's
 * input norms feed q/k/v/gate/up). For each row m of X (d = Kin values):
 *   S = sum_k x_k^2 computed exactly (fp16 squares are integer multiples of
 *       2^-48; the sum is held in 128 bits), rounded once to fp32 (to
 *       nearest, ties to even);
 *   ms = S / d; r = 1 / sqrt(ms + eps), r = 0 when ms + eps == 0;
 *   t_k = fp16(x_k * r); y_k = fp16(t_k * w_k) (each step one correctly
 *   rounded operation);
 *   then the codes and scale of y as p4q_quant_act.
 *   X [M, Kin] fp16, rows ldx elements apart (device, read); finite values
 *   w [Kin] fp16 gain (device, read); y must stay finite
 *   eps >= 0
 *   Xq [M, Kin/2], s_a [M]           written
 *   Xu [M, Kin], sum_xu [M]          the expanded codes (p4q_expand_codes
 *                                    form) or both NULL
 * Requires M >= 0, 16 <= Kin <= P4Q_MAX_ROW, Kin % 16 == 0, ldx >= Kin,
 * ldx % 8 == 0, 16-byte aligned pointers. M == 0 is a no-op. */
p4q_status p4q_rmsnorm_quant_expanded(const uint16_t* X, int ldx, const uint16_t* w, float eps, int M, int Kin,
                                      uint8_t* Xq, float* s_a, uint8_t* Xu, int32_t* sum_xu, p4q_stream_t stream);

/* Causal softmax attention on the pruned sequence with FP16 keys and values
 * (App. B: the decoder's linears run in W4A4 while the key and value caches
 * stay in FP16). For each sample b of m positions, head h and position i:
 *   o_i = sum_{j <= i} p_ij v_j, p_i. = softmax_j(q_i . k_j / sqrt(dh)),
 * with key/value head h / (H / Hkv). Position encodings are applied by the
 * caller. fp16 inputs, products accumulated in fp32, p rounded to fp16 before
 * the product with v (keys taken 128 at a time with running row maxima: p is
 * relative to a reference maximum of the keys so far, which moves when a
 * chunk's maximum exceeds it by 2^8 in p, the earlier partial sums and
 * products rescaled then), fp32 row sums, fp16 output.
 *   q [B*m, ldq] fp16: row b*m + i holds position i of sample b, head h in
 *                      columns h*dh .. h*dh + dh - 1   (device, read)
 *   k, v [B*m, ldk / ldv] fp16, Hkv heads likewise   (device, read; rows may
 *                      be column blocks of a fused projection output)
 *   o [B*m, ldo] fp16, columns 0 .. H*dh - 1 written (device)
 * Requires dh == 128, 1 <= m <= 8192, H % Hkv == 0, ld >= the row's heads *
 * dh, every ld % 8 == 0, 16-byte aligned pointers. B == 0 is a no-op. */
p4q_status p4q_causal_attention(const uint16_t* q, int ldq, const uint16_t* k, int ldk, const uint16_t* v, int ldv,
                                int B, int m, int H, int Hkv, int dh, uint16_t* o, int ldo, p4q_stream_t stream);

/* ---------------------------------------------------------------------- */
/* Pruning-aware calibration data path (Sec. 3.3, Eq. 5; App. A, Eq. 9)     */
/* ---------------------------------------------------------------------- */

/* Workspace of p4q_block_mse for B samples (fp64 partial sums); 0 when B is
 * outside 1 .. 1024. */
size_t p4q_block_mse_workspace_bytes(int B);

/* Eq. 5's block objective. Sample n owns rows offsets[n] .. offsets[n+1]-1 of
 * the W4A4 block output Yq and of the full-precision block output Yf (both
 * computed on the same pruned input H^{FP,keep}, e.g. the X of
 * p4q_select_gather_quant):
 *   e[n] = ||Yq_n - Yf_n||_F^2 / (m_n d),   *L = (1/B) sum_n e[n].
 * Squares summed in fp32 per thread over a few hundred values, combined in
 * fp64 in a fixed order (the result does not depend on the launch).
 *   Yq, Yf  [offsets[B], ld] fp16 (device, read), d columns used
 *   offsets HOST array of B + 1 ints, offsets[0] = 0, strictly increasing
 *   e [B], L [1] fp32 (device, written)
 *   ws      device workspace of p4q_block_mse_workspace_bytes(B) bytes
 * Requires 1 <= B <= 1024, d % 8 == 0, ld >= d, ld % 8 == 0, 16-byte aligned
 * Yq, Yf and ws. */
p4q_status p4q_block_mse(const uint16_t* Yq, int ldq, const uint16_t* Yf, int ldf, const int32_t* offsets, int B,
                         int d, float* e, float* L, void* ws, size_t ws_bytes, p4q_stream_t stream);

/* Eq. 9's Top-K replacement ratio per sample: the Top-K sets of the scores
 * of the same N tokens under a reference and an alternative precision (the K
 * largest scores; ties, with -0 equal to +0, to the lower index) and
 *   inter[b] = |T_ref & T_alt|,   rho[b] = fl32(1 - fl32(inter[b] / K)).
 *   s_ref, s_alt [B, N] fp32 finite (device, read)
 *   inter [B] int32, rho [B] fp32 (device, written)
 * Requires 1 <= K <= N <= P4Q_MAX_TOKENS, 0 <= B <= 65535 (0: no-op). */
p4q_status p4q_topk_replacement(const float* s_ref, const float* s_alt, int B, int N, int K, int32_t* inter,
                                float* rho, p4q_stream_t stream);

/* Per-output-channel weight quantization (App. B.3: symmetric, per output
 * channel, then round-to-nearest): the same per-row quantizer applied to each
 * output row of W.
 *   W   [N, Kin] fp16 row-major, one row per output channel (device, read)
 *   Wq  [N, Kin/2] packed INT4 (device, written)
 *   s_w [N] fp32 (device, written)
 * Same size limits as p4q_quant_act. Not on the timed path (offline). */
p4q_status p4q_quant_weight(const uint16_t* W, int N, int Kin, uint8_t* Wq, float* s_w,
                            p4q_stream_t stream);

/* ---------------------------------------------------------------------- */
/* W4A4 linear (App. B.3: INT4 weights per output channel, INT4 activations */
/* per token)                                                              */
/* ---------------------------------------------------------------------- */

/* Y[m,n] = fp16_rne( ((float)acc[m,n] * s_a[m]) * s_w[n] ),
 * acc[m,n] = sum_k code_x[m,k] * code_w[n,k] computed exactly (int32).
 *   Xq  [M, Kin/2] packed INT4, s_a [M] fp32   (device, read)
 *   Wq  [N, Kin/2] packed INT4, s_w [N] fp32   (device, read)
 *   Y   [M, N] fp16 row-major                  (device, written)
 * Requires M >= 0, N >= 1, Kin % 128 == 0, 128 <= Kin <= P4Q_MAX_ROW,
 * N % 8 == 0. Runs on the tcgen05 tensor cores. */
p4q_status p4q_w4a4_linear(const uint8_t* Xq, const float* s_a, int M, int Kin,
                           const uint8_t* Wq, const float* s_w, int N, uint16_t* Y,
                           p4q_stream_t stream);

/* Test entry: the exact int32 accumulators of the same integer matmul,
 * acc [M, N] int32 row-major (device, written). Same limits as above. */
p4q_status p4q_w4a4_gemm_s32(const uint8_t* Xq, int M, int Kin, const uint8_t* Wq, int N,
                             int32_t* acc, p4q_stream_t stream);

/* Workspace bytes for p4q_w4a4_linear_ws / p4q_w4a4_gemm_s32_ws on an
 * M x N x Kin linear: both operands as one byte per code plus their row
 * sums. 0 for sizes the linear rejects. */
size_t p4q_w4a4_linear_workspace_bytes(int M, int N, int Kin);

/* p4q_w4a4_linear with a caller workspace (App. B.3; same results bit for
 * bit). With a workspace, large linears (M >= 512 and N >= 256) first expand
 * both packed operands into it, one byte per code (u = v + 8) with the row
 * sums of u, and then run a GEMM whose operands reach the tensor cores by
 * TMA alone (no unpacking on the SMs that run the MMAs); other shapes, or
 * ws == NULL, run exactly as p4q_w4a4_linear. The paper has no counterpart:
 * this is a deployment choice for GPUs without 4-bit integer MMAs.
 *   ws        device workspace, 16-byte aligned, or NULL
 *   ws_bytes  >= p4q_w4a4_linear_workspace_bytes(M, N, Kin) when ws != NULL,
 *             else P4Q_ERR_WORKSPACE_TOO_SMALL (P4Q_ERR_MISALIGNED if unaligned)
 * The workspace is scratch overwritten by every call: calls sharing one must
 * be ordered (same stream). Other arguments and rules as p4q_w4a4_linear. */
p4q_status p4q_w4a4_linear_ws(const uint8_t* Xq, const float* s_a, int M, int Kin, const uint8_t* Wq,
                              const float* s_w, int N, uint16_t* Y, void* ws, size_t ws_bytes,
                              p4q_stream_t stream);

/* The two halves of the expanded-operand path, for callers that expand an
 * operand once and use it in several linears (activations shared by the q,
 * k, v, gate and up projections) or keep expanded weights.
 * p4q_expand_codes: packed INT4 rows q [rows, Kin/2] -> u [rows, Kin] bytes,
 * u = v + 8 for each code v (per packed 32-bit word: its four low-nibble
 * codes, then its four high-nibble codes), and sum_u [rows] int32.
 *   Kin % 128 == 0, Kin <= P4Q_MAX_ROW; 16-byte aligned pointers; rows == 0 is a no-op.
 * p4q_w4a4_linear_expanded: Y = fp16_rne(((float)acc * s_a[m]) * s_w[n]) with
 * acc the exact integer dot product of the codes, from expanded operands
 * (Xu, sum_xu: [M, Kin], [M]; Wu, sum_wu: [N, Kin], [N]); same results as
 * p4q_w4a4_linear. Requires N >= 256, N % 8 == 0, Kin % 128 == 0. */
p4q_status p4q_expand_codes(const uint8_t* q, int rows, int Kin, uint8_t* u, int32_t* sum_u, p4q_stream_t stream);
p4q_status p4q_w4a4_linear_expanded(const uint8_t* Xu, const int32_t* sum_xu, const float* s_a, int M, int Kin,
                                    const uint8_t* Wu, const int32_t* sum_wu, const float* s_w, int N, uint16_t* Y,
                                    p4q_stream_t stream);

/* p4q_w4a4_linear_expanded that also records, for nblk <= 2 column blocks
 * of Y, each row's abs-max over the block as the fp16 bit pattern the
 * per-token quantizer of the next linear reads first (App. A: per-token
 * activations; the block is that linear's input, e.g. the q or up part of a
 * fused q|k|v|gate|up output):
 *   rowmax[b * M + m] = max over c in [col0[b], col0[b] + ncols[b]) of
 *                       (bits(Y[m, c]) & 0x7FFF)
 * (non-negative fp16 values order as their bit patterns). The call clears
 * rowmax on `stream`, then the GEMM's epilogue takes the maxima with one
 * atomic per row and tile. Y and every other output as
 * p4q_w4a4_linear_expanded. The paper has no counterpart.
 *   col0, ncols  host arrays of nblk entries, multiples of 32,
 *                col0[b] + ncols[b] <= N
 *   rowmax       [nblk, M] uint32 (device, written), 16-byte aligned */
p4q_status p4q_w4a4_linear_expanded_rowmax(const uint8_t* Xu, const int32_t* sum_xu, const float* s_a, int M,
                                           int Kin, const uint8_t* Wu, const int32_t* sum_wu, const float* s_w, int N,
                                           uint16_t* Y, int nblk, const int* col0, const int* ncols,
                                           uint32_t* rowmax, p4q_stream_t stream);

/* p4q_quant_act_expanded of nblk <= 2 column blocks of Y [M, ldy] fp16
 * (block b: columns col0[b] .. col0[b] + ncols[b] - 1) whose row abs-max is
 * given (rowmax as p4q_w4a4_linear_expanded_rowmax writes it): the same
 * codes, scales, expanded codes and row sums bit for bit, in one streaming
 * pass over both blocks (no abs-max pass). The paper has no counterpart.
 *   Xq[b]   [M, ncols[b]/2] packed INT4, or Xq == NULL / Xq[b] == NULL to
 *           skip the packed form (device, written)
 *   s_a[b]  [M] fp32; Xu[b] [M, ncols[b]] bytes; sum_xu[b] [M] int32
 *           (device, written)
 *   col0, ncols and the pointer arrays are host arrays of nblk entries.
 * Requires ncols[b] % 256 == 0, ncols[b] <= P4Q_MAX_ROW, col0[b] % 8 == 0,
 * col0[b] + ncols[b] <= ldy, ldy % 8 == 0, 16-byte aligned pointers. M == 0
 * is a no-op. */
p4q_status p4q_quant_act_expanded_rowmax(const uint16_t* Y, int ldy, int M, int nblk, const int* col0,
                                         const int* ncols, const uint32_t* rowmax, uint8_t* const* Xq,
                                         float* const* s_a, uint8_t* const* Xu, int32_t* const* sum_xu,
                                         p4q_stream_t stream);

/* Test view of the same path: the exact int32 accumulators (as
 * p4q_w4a4_gemm_s32). */
p4q_status p4q_w4a4_gemm_s32_ws(const uint8_t* Xq, int M, int Kin, const uint8_t* Wq, int N, int32_t* acc,
                                void* ws, size_t ws_bytes, p4q_stream_t stream);

/* ---------------------------------------------------------------------- */
/* Quantization-aware visual-token selector (Sec. 3.2, Eq. 4)               */
/* ---------------------------------------------------------------------- */

/* CLS-to-patch saliency A_cls, the input of the selector's stage 2 (Sec. 3.2,
 * Visual Saliency: in the vision tower's final self-attention layer each
 * crop's [CLS] token is the query; the attention weights of the patch keys
 * are averaged across the heads). Per image b, crop c and head h:
 *   l_0 = q . k_cls / sqrt(dh), l_i = q . k_i / sqrt(dh) for the crop's
 *   patches i; p = softmax over {l_0, l_i} (the CLS key is part of the
 *   attention row); A_cls[b, i] = (1 / H) sum_h p_i.
 * fp16 inputs, fp32 arithmetic (products accumulated in fp32, expf, one
 * division per head), heads summed in order (deterministic).
 *   q_cls [B, C, H, dh] fp16  final-layer CLS query of each crop, per head
 *   k_cls [B, C, H, dh] fp16  final-layer CLS key of each crop, per head
 *   k     [B, N, H, dh] fp16  patch keys; crop c holds tokens
 *                             [c * N / C, (c + 1) * N / C)
 *   A_cls [B, N] fp32         written
 * Requires 1 <= B <= 65535, 1 <= C, N % C == 0, 1 <= N / C <= P4Q_MAX_TOKENS,
 * dh in {32, 64, 80, 128}, 1 <= H <= 32, H * (N / C) * 4 <= 227 KB (one
 * crop's weights in shared memory), 16-byte aligned pointers. All device
 * pointers; asynchronous on `stream`. */
p4q_status p4q_cls_saliency(const uint16_t* q_cls, const uint16_t* k_cls, const uint16_t* k, int B, int N, int C,
                            int H, int dh, float* A_cls, p4q_stream_t stream);

/* Device workspace needed by p4q_select / p4q_select_gather_quant for these
 * sizes (bytes, a multiple of 256). Returns 0 if the sizes are invalid. */
size_t p4q_select_workspace_bytes(int B, int N, int d, int J, const p4q_select_params* params);

/* Selects K of the N visual tokens of each image (Sec. 3.2, Eq. 4):
 *   - V and Q are fake-quantized per row with the 4-bit quantizer above
 *     (the selector sees only the fake-quantized copies);
 *   - CosSim(a, b) of fake-quantized rows is evaluated on their codes as
 *     (float)dot / sqrtf((float)|c_a|^2 * (float)|c_b|^2), fp32, 0 if a norm
 *     is 0 (the positive scales cancel);
 *   - stage 1 (query relevance): concept j = 0..J-1 in turn keeps its
 *     floor(K_q/J) + (j < K_q % J) best-cosine tokens not kept yet;
 *   - stage 2 (visual saliency): the K_s largest A_cls among tokens not kept;
 *   - stage 3 (visual diversity): K_d times, keep the token whose largest
 *     cosine to the kept set is smallest (the first token when nothing is kept);
 *   - every tie goes to the lower token index.
 *   V     [B, N, d] fp16 projector features (device, read)
 *   Q     [B, J, d] fp16 concept embeddings, or NULL (then J is ignored)
 *   A_cls [B, N] fp32 CLS-to-patch attention (head-averaged), or NULL
 *   idx   [B, K] int32, kept token indices in ascending order (device, written)
 *   ws    device workspace of at least p4q_select_workspace_bytes() bytes,
 *         256-byte aligned; its contents are scratch.
 * Requires 1 <= B, 1 <= K <= N <= P4Q_MAX_TOKENS, 0 <= J <= P4Q_MAX_CONCEPTS,
 * d % 128 == 0, 128 <= d <= P4Q_MAX_ROW, 0 <= alpha, beta and
 * alpha + beta <= 1000.
 * All work is ordered on `stream`. For images of at most 1024 tokens with a
 * diversity stage (K_d > 0) the GEMM of all token pairs runs beside the
 * stage 1-2 launch on a second stream the library owns
 * (one per device, created on the first call that is not being captured into
 * a CUDA graph; until then the order is serial), forked from and joined back
 * into `stream` by events inside the call, so a graph captured from `stream`
 * contains both branches; a host lock keeps concurrent callers' fork/join
 * pairs apart. */
p4q_status p4q_select(const uint16_t* V, int B, int N, int d, const uint16_t* Q, int J,
                      const float* A_cls, const p4q_select_params* params, int32_t* idx,
                      void* ws, size_t ws_bytes, p4q_stream_t stream);

/* p4q_select for callers that cannot allocate device memory when they select
 * (a fixed memory budget set at start-up, a plugin inside a runtime that owns
 * the allocator): same inputs, outputs and results as p4q_select, without the
 * workspace arguments. The paper has no counterpart; this is a deployment
 * convenience of this library.
 *
 * Scratch: a fixed array of P4Q_NOALLOC_SCRATCH_BYTES inside the library's
 * device image (enough for at least 8 images of 576 x 4096 with 3 concepts
 * and K = 192). Sizes whose workspace for this call exceeds it return
 * P4Q_ERR_WORKSPACE_TOO_SMALL and launch nothing. Each call looks up the
 * array's device address in the current context (cudaGetSymbolAddress), so
 * it stays right after cudaDeviceReset or in another context. Under CUDA's
 * lazy module loading the array is committed on a device by the first call
 * there (which may then fail with P4Q_ERR_CUDA on a full device): make that
 * first call at start-up, inside the caller's memory budget, and before any
 * stream capture. The call allocates nothing itself and creates no stream or
 * event (its launches run in order on `stream`). All calls on a device
 * share the one array, which keeps the last call's contents (every region is
 * written before it is read, so nothing needs clearing): calls whose work
 * overlaps on the GPU (other streams, or several host threads) race and give
 * undefined results, so serialize them. */
#define P4Q_NOALLOC_SCRATCH_BYTES (48u << 20)
p4q_status p4q_select_noalloc(const uint16_t* V, int B, int N, int d, const uint16_t* Q, int J,
                              const float* A_cls, const p4q_select_params* params, int32_t* idx,
                              p4q_stream_t stream);

/* The selector followed by the gather of the original FP16 features of the
 * kept tokens (Sec. 3.2: the fake-quantized copies only decide the indices)
 * and the per-token INT4 quantization of the pruned sequence for the first
 * W4A4 linear. Per image b the pruned sequence is
 *   X[b] = [ V[b, idx[b,0]], ..., V[b, idx[b,K-1]], text[b,0], ..., text[b,T-1] ]
 *   text [B, T, d] fp16 (device, read), or NULL when T == 0
 *   idx  [B, K] int32 ascending (device, written)
 *   X    [B, K+T, d] fp16 (device, written)
 *   Xq   [B*(K+T), d/2] packed INT4, s_a [B*(K+T)] fp32 (device, written):
 *        the activation quantizer of p4q_quant_act applied to every row of X.
 * Other arguments and limits as p4q_select; T >= 0. */
p4q_status p4q_select_gather_quant(const uint16_t* V, int B, int N, int d, const uint16_t* Q,
                                   int J, const float* A_cls, const uint16_t* text, int T,
                                   const p4q_select_params* params, int32_t* idx, uint16_t* X,
                                   uint8_t* Xq, float* s_a, void* ws, size_t ws_bytes,
                                   p4q_stream_t stream);

/* p4q_select_gather_quant that also writes the pruned sequence's codes in
 * the expanded form of p4q_expand_codes (Xu [B*(K+T), d] bytes, sum_xu
 * [B*(K+T)] int32; both NULL or both set), for p4q_w4a4_linear_expanded,
 * without a second pass over the codes. With Xu set, Xq may be NULL (only
 * the expanded form is written). The paper has no counterpart. */
p4q_status p4q_select_gather_quant_expanded(const uint16_t* V, int B, int N, int d, const uint16_t* Q, int J,
                                            const float* A_cls, const uint16_t* text, int T,
                                            const p4q_select_params* params, int32_t* idx, uint16_t* X,
                                            uint8_t* Xq, float* s_a, uint8_t* Xu, int32_t* sum_xu, void* ws,
                                            size_t ws_bytes, p4q_stream_t stream);

#ifdef __cplusplus
}
#endif

#endif /* P4Q_H_ */
