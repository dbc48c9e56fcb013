// Host-side declarations shared by the translation units of libp4q.so.
#pragma once

#include <cstddef>
#include <cstdint>
#include <cuda.h>
#include <cudaTypedefs.h>
#include <cuda_runtime.h>

#include <utility>

namespace p4q {

// Launches kernel<<<grid, block, smem, stream>>>(args...) with programmatic
// stream serialization (see pdl_wait in p4q_device.cuh).
template <typename... KArgs, typename... Args>
cudaError_t launch_pdl(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem, cudaStream_t stream,
                       Args&&... args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = stream;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, kernel, std::forward<Args>(args)...);
}


// ------------------------------------------------------------ quantizer
// Row source for the per-row quantizer: either a dense [rows, L] fp16 matrix,
// or the pruned sequence of the selector (kept visual rows, then text rows).
struct RowSource {
  const uint16_t* X = nullptr;     // dense source, or V [B, N, L] when idx != nullptr
  long long ldx = 0;               // dense mode: elements between rows (0: L)
  const int32_t* idx = nullptr;    // [B, K] kept indices (gather mode)
  const uint16_t* text = nullptr;  // [B, T, L] (gather mode)
  int N = 0, K = 0, T = 0;         // gather mode sizes
  const uint16_t* X2 = nullptr;    // dense rows split, split + 1, ... (the second sinks; dense mode)
  int split = 0;
};

// Outputs of the per-row quantizer. Optional pointers may be null.
struct RowSinks {
  uint8_t* codes = nullptr;   // [rows, L/2] packed INT4 (may be null when u is given)
  float* scale = nullptr;     // [rows] (required)
  int32_t* norm2 = nullptr;   // [rows] sum of squared codes
  uint16_t* copy = nullptr;   // [rows, L] fp16 copy of the source row (gather mode)
  uint8_t* u = nullptr;       // [rows, L] codes expanded to one byte each (u = v + 8, the GEMM's order)
  int32_t* sum_u = nullptr;   // [rows] sum of u (with u)
};

// Rows at or past src.split (when src.X2 is set) come from X2 and go to
// *out2, renumbered from 0: two row sets quantized by one launch.
cudaError_t launch_quant_rows(const RowSource& src, int rows, int L, const RowSinks& out,
                              cudaStream_t stream, const RowSinks* out2 = nullptr);

// Per-token quantizer of up to two column blocks of Y [M, ldy] fp16 whose
// rows' abs-max is known (fp16 bit patterns rowmax [nblk, M], as the GEMM's
// row-max epilogue writes them): the codes, scales and expanded codes of
// launch_quant_rows, one streaming pass (one warp per block row).
struct RowmaxBlock {
  int col0 = 0, L = 0;        // columns col0 .. col0 + L of Y (L % 256 == 0)
  uint8_t* codes = nullptr;   // [M, L/2] or null
  float* scale = nullptr;     // [M]
  uint8_t* u = nullptr;       // [M, L]
  int32_t* sum_u = nullptr;   // [M]
};
cudaError_t launch_quant_rowmax(const uint16_t* Y, int ldy, int M, int nblk, const RowmaxBlock* blk,
                                const uint32_t* rowmax, cudaStream_t stream);

// The selector's token pass: V [B, N, d] fake-quantized per row into out's
// scale, norm2, u and sum_u (all required), and, for J > 0, the exact code
// dot products with the image's J concepts (expanded codes qu [B, J, d], row
// sums qsum [B, J]) as floats qdots [B * N, qp]. For d % 256 == 0, d <=
// kTokenQuantMaxRow and J * d <= 96 KB (select_token_quant_applies).
constexpr int kTokenQuantMaxRow = 5120;
bool select_token_quant_applies(int d, int J);
cudaError_t launch_select_token_quant(const uint16_t* V, int B, int N, int d, int J, const uint8_t* qu,
                                      const int32_t* qsum, const RowSinks& out, float* qdots, int qp,
                                      cudaStream_t stream);

// ------------------------------------------------------------ GEMM
enum class GemmOut { kHalf = 0, kS32 = 1, kCos = 2 };

struct GemmArgs {
  const uint8_t* A = nullptr;  // [batch, M, K/2] packed INT4
  const uint8_t* B = nullptr;  // [batch, N, K/2] packed INT4
  int M = 0, N = 0, K = 0, batch = 1;
  long long a_batch_stride = 0;  // rows between batches of A (0 for batch 1)
  long long b_batch_stride = 0;
  GemmOut out = GemmOut::kHalf;
  void* D = nullptr;              // [batch, M, d_pitch] fp16 / int32 / fp32
  int d_pitch = 0;                // output row pitch in elements (0 = N); pitch * size % 16 == 0
  const float* s_a = nullptr;     // kHalf: [M]
  const float* s_b = nullptr;     // kHalf: [N]
  const int32_t* norm_a = nullptr;  // kCos: [batch, M] squared code norms
  const int32_t* norm_b = nullptr;  // kCos: [batch, N]
  int tile_n = 256;                 // expanded-operand int32 tiles: columns per tile (multiple of 32, <= 256)
  bool f32_out = false;             // expanded-operand int32 tiles: the exact integers as fp32 values
  // expanded-operand fp16 output: per row, the largest |Y| bit pattern over
  // each of rm_n <= 2 column ranges [rm_c0, rm_c1) (multiples of 32), into
  // rowmax [rm_n, M] by atomicMax (cleared by the caller first)
  uint32_t* rowmax = nullptr;
  int rm_n = 0;
  int rm_c0[2] = {0, 0}, rm_c1[2] = {0, 0};
};

// Returns cudaSuccess or the launch error; sets *unsupported when the shape
// cannot run on this kernel.
cudaError_t launch_w4a4_gemm(const GemmArgs& g, cudaStream_t stream);

// W4A4 linear / int32 accumulators for M <= 8 rows (decode): streams the
// packed weights, dp4a against the activation rows staged in shared memory.
bool gemv_applies(const GemmArgs& g);
cudaError_t launch_gemv(const GemmArgs& g, cudaStream_t stream);

// Which GEMM kernel serves fp16 / int32 outputs: -1 automatic (the
// weight-streaming kernel for M <= 8, the CTA-pair kernel for large fp16
// linears), 0 single-CTA only, 1 CTA-pair whenever the shape allows (N >= 256).
void set_gemm_pair_mode(int mode);
// Expanded-operand path: 0 automatic (M >= 512), 1 never, 2 whenever a workspace is given.
void set_gemm8_mode(int mode);

// ------------------------------------------------------------ SwiGLU -> quantizer
// Rows of gate / up (fp16, row pitches ldg / ldu in elements): codes of
// h = silu(gate) * up per row (packed; expanded + row sums when Xu != null).
cudaError_t launch_swiglu_quant(const uint16_t* gate, long long ldg, const uint16_t* up, long long ldu, int M, int K,
                                uint8_t* Xq, float* s_a, uint8_t* Xu, int32_t* sum_xu, cudaStream_t stream);

// ------------------------------------------------------------ RMSNorm -> quantizer
// Rows of X (fp16, row pitch ldx elements), gain w [K] fp16: codes of the
// RMSNorm of each row (packed; expanded + row sums when Xu != null).
cudaError_t launch_rmsnorm_quant(const uint16_t* X, long long ldx, const uint16_t* w, float eps, int M, int K,
                                 uint8_t* Xq, float* s_a, uint8_t* Xu, int32_t* sum_xu, cudaStream_t stream);

// ------------------------------------------------------------ causal attention (FP16 K/V)
// Longest sample the kernel takes (the keys stream through in chunks of 128).
constexpr int kAttnMaxLen = 8192;
// Dynamic shared memory of one CTA for samples of m positions.
size_t causal_attention_smem_bytes(int m);
// q [B*m, ldq], k / v [B*m, ldk / ldv], o [B*m, ldo] fp16 rows; head dim 128.
cudaError_t launch_causal_attention(const uint16_t* q, long long ldq, const uint16_t* k, long long ldk,
                                    const uint16_t* v, long long ldv, int B, int m, int H, int Hkv, uint16_t* o,
                                    long long ldo, cudaStream_t stream);
unsigned int attn_read_and_clear_error();

// ------------------------------------------------------------ calibration data path
constexpr int kMseMaxSamples = 1024;
// CTAs per sample of the block-objective reduction, and its workspace (fp64 partials).
int block_mse_chunks(int B);
size_t block_mse_workspace_bytes(int B);
// off: host array of B + 1 row offsets (validated by the caller).
cudaError_t launch_block_mse(const uint16_t* Yq, long long ldq, const uint16_t* Yf, long long ldf, const int32_t* off,
                             int B, int d, double* partial, float* e, float* L, cudaStream_t stream);
// Top-K sets of two score rows per sample and their intersection (selector's radix select).
cudaError_t launch_topk_replacement(const float* s_ref, const float* s_alt, int B, int N, int K, int32_t* inter,
                                    float* rho, cudaStream_t stream);

// ------------------------------------------------------------ CLS saliency
// Shared memory of one (image, crop) CTA: H x (N / C) fp32 weights.
size_t cls_saliency_smem_bytes(int N, int C, int H);
// Heads one CTA takes for this head dimension (one warp each).
int cls_saliency_max_heads(int dh);
// dh in {32, 64, 80, 128}; else cudaErrorInvalidValue.
cudaError_t launch_cls_saliency(const uint16_t* q_cls, const uint16_t* k_cls, const uint16_t* k, int B, int N,
                                int C, int H, int dh, float* A, cudaStream_t stream);

// ------------------------------------------------------------ selector
struct SelectPlan {
  int B, N, d, J, K, Kq, Ks, Kd;
};

struct SelectWorkspace {
  float* vscale;     // [B*N]
  int32_t* vnorm;    // [B*N]
  uint8_t* qcodes;   // [B*J, d/2]
  uint8_t* qu;       // [B*J, d] the concepts' codes, one byte each (u = v + 8)
  int32_t* qsum;     // [B*J] sum of those bytes
  float* qscale;     // [B*J]
  int32_t* qnorm;    // [B*J]
  float* qdots;      // [B, N, q_pitch] code dot products of every token with its image's concepts (exact, fp32)
  int q_pitch;       // J rounded up to a multiple of 4
  uint8_t* vu;       // [B*N, d] codes, one byte each (u = v + 8)
  int32_t* vsum;     // [B*N] sum of those bytes
  uint32_t* kept12;  // [B, ceil(N/32)] kept set after stages 1-2, as bits
  int32_t* r0tok;    // [B, R0] that kept set, ascending (R0 = Kq + Ks)
  uint8_t* r0u;      // [B, R0, d] its expanded codes
  int32_t* r0sum;    // [B, R0]
  int32_t* r0norm;   // [B, R0]
  float* dots;       // [B, N, dot_pitch] code dot products of every token with every token of R0 (exact,
                     // fp32), for R0 > kCosMaxCols
  float* mpart;      // [r0_parts, B, N] each token's largest cosine per column tile of R0 (r0_parts > 1)
  int r0_parts;      // column tiles of the R0 GEMM (cosine-max epilogue), else 0
  int dot_pitch;     // R0 rounded up to a multiple of 4
  int r0_tile_n;     // column tile width of that GEMM
  float* m;          // [B, N] the largest cosine of each token to R0 (stage 3's initial m)
  int C;             // candidates of stage 3 per image (0 without a diversity stage)
  int32_t* cand;     // [B, C] the candidates, ascending
  uint8_t* candu;    // [B, C, d] their expanded codes
  int32_t* candsum;  // [B, C]
  int32_t* candnorm; // [B, C]
  float* cdots;      // [B, C, cpitch] their code dot products (exact, fp32)
  int cpitch;        // C rounded up to a multiple of 4
  bool gram;         // small images: every token is a candidate (C = N, cdots by token, no cand lists)
};

// Candidates of stage 3: up to kCandExtra more than the K_d picks (a pool's
// worth), at most kCandMax. Images of at most kGramMaxTokens tokens take every
// token as a candidate: one GEMM of all their token pairs replaces R0's GEMM,
// the candidate selection and the gather (Gram mode).
constexpr int kCandExtra = 128, kCandMax = 1024, kGramMaxTokens = 1024;
// Kept sets of at most kCosMaxCols tokens take their tokens' cosine maxima
// from one GEMM with a cosine-max epilogue (a partial maximum per column tile,
// merged by the candidate selection); larger ones from an int32-tile GEMM and
// a row pass.
constexpr int kCosMaxCols = 1024;
bool select_gram_mode(int N, int Kd);
int select_candidates(int N, int R0, int Kd);

// Workspace of one selector call with R0 = Kq + Ks tokens after stages 1-2
// and C candidates in stage 3 (Gram mode: C = N). Every region grows with R0
// and with C, so the layout at the largest R0 and C covers any call.
size_t select_workspace_layout(int B, int N, int d, int J, int R0, int C, bool gram, SelectWorkspace* ws,
                               void* base);
int r0_tile_n(int R0);

// Stages 1-2: kept12 bits, r0tok, and idx when p.Kd == 0.
// qdots on the expanded-operand CTA-pair GEMM (tokens as A rows, the image's
// concepts as B rows, one 32-column tile).
cudaError_t launch_query_dots(const SelectPlan& p, const SelectWorkspace& ws, cudaStream_t stream);
cudaError_t launch_select_stages12(const SelectPlan& p, const SelectWorkspace& ws, const float* A_cls, int32_t* idx,
                                   cudaStream_t stream);
cudaError_t launch_gather_r0(const SelectPlan& p, const SelectWorkspace& ws, cudaStream_t stream);
// m[b, i] = max over the R0 tokens r of cos(i, r): the exact dot products on
// the expanded-operand CTA-pair GEMM (tokens as A rows, R0 as B rows, int32
// tiles), then their cosines and maxima by a full-GPU row pass.
cudaError_t launch_r0_cosmax(const SelectPlan& p, const SelectWorkspace& ws, cudaStream_t stream);
// The candidates of stage 3 (per image), their expanded codes, and the
// code dot products of every pair of them (a batched tensor-core GEMM).
cudaError_t launch_candidates(const SelectPlan& p, const SelectWorkspace& ws, cudaStream_t stream);
// Gram mode: the code dot products of every token pair of each image into
// cdots; then each token's largest cosine to R0 from them (m).
cudaError_t launch_gram(const SelectPlan& p, const SelectWorkspace& ws, cudaStream_t stream);
cudaError_t launch_gram_cosmax(const SelectPlan& p, const SelectWorkspace& ws, cudaStream_t stream);
// Stage 3 (greedy max-min diversity) from kept12, m and the candidates; writes idx.
cudaError_t launch_select_diverse(const SelectPlan& p, const SelectWorkspace& ws, int32_t* idx, cudaStream_t stream);
unsigned int diverse_read_and_clear_error();

// Device error words of the kernels with bounded waits (GEMMs, quantizer).
unsigned int gemm_read_and_clear_error();
unsigned int gemm8_read_and_clear_error();
unsigned int quant_read_and_clear_error();

// ------------------------------------------------------------ shared GEMM helpers (p4q_gemm.cu)
int num_sms();
// 3-D map over the output [batch][rows][cols] with row pitch `pitch` elements;
// 32 x 32 boxes in the swizzle the epilogues write.
bool make_output_map(CUtensorMap* map, void* base, GemmOut out, int rows, int cols, int pitch, int batch);
PFN_cuTensorMapEncodeTiled_v12000 get_encode_fn();

// ------------------------------------------------------------ expanded-operand GEMM (p4q_gemm8.cu)
// Bytes of the workspace the expanded-operand path needs for an M x N x K
// linear: both operands as one byte per code (u = v + 8) and their row sums.
size_t gemm8_workspace_bytes(int M, int N, int K);
// Whether the expanded-operand path serves this shape (large enough that the
// expansion pays for itself).
bool gemm8_applies(const GemmArgs& g);
// Expands both operands into the workspace, then runs the FP8 GEMM.
cudaError_t launch_w4a4_gemm8(const GemmArgs& g, void* ws, size_t ws_bytes, cudaStream_t stream);
// The two halves: packed rows -> one byte per code (u = v + 8) + row sums of u;
// the GEMM on expanded operands (g.A / g.B unused; batch 1, N >= 256).
cudaError_t launch_expand_codes(const uint8_t* q, int rows, int K, uint8_t* u, int32_t* sum_u, cudaStream_t stream);
cudaError_t launch_gemm8(const GemmArgs& g, const uint8_t* a8, const int32_t* sum_a, const uint8_t* b8,
                         const int32_t* sum_b, cudaStream_t stream);

// Throughput probes of the integer contraction pipes (roofline denominators):
// kind 0 tcgen05 kind::f8f6f4 MMAs, 1 mma.sync m16n8k32 s8, 2 dp4a; *ops is the
// number of integer (or FP8) operations the launch performs.
cudaError_t launch_peak_probe(int kind, int iters, uint32_t* sink, double* ops, cudaStream_t stream);
size_t peak_probe_sink_words();
unsigned int peak_read_and_clear_error();

// One bounded wait that nothing completes: times out after limit_ns and sets
// the GEMM's device error word (tests the time-out path).
cudaError_t launch_expired_wait(unsigned long long limit_ns, cudaStream_t stream);

}  // namespace p4q
