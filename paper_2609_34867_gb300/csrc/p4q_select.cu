// Quantization-aware visual-token selector (Sec. 3.2, Eq. 4 of the paper):
// query relevance and saliency stages, and the operand preparation of the
// diversity stage (p4q_diverse.cu runs the greedy rounds).
//
// Inputs are the fake-quantized copies produced by the quantizers (the codes
// of every visual token and concept expanded to one byte each, u = v + 8,
// with their row sums, and the squared code norms) and the exact code dot
// products of every token with its image's concepts (from the token pass, or
// a narrow tensor-core GEMM). The cosine of two fake-quantized rows is
// evaluated on their codes (code_cosine: the positive per-row scales cancel).
//
// Kernels:
//   select_stages12_kernel  one CTA per image, one thread per 4 tokens: stage 1
//                           (per-concept top quota), stage 2 (CLS-saliency top
//                           K_s); writes the kept set R0 as bits and as an
//                           ascending token list (and as idx when K_d = 0).
//   gather_rows_kernel      the expanded codes, row sums and norms of listed
//                           tokens (R0, or the diversity candidates), row by
//                           row, as an operand of the tensor-core GEMMs.
//   r0_cosmax_kernel        each token's largest cosine to R0 from exact dot
//                           products in fp32 rows: the token-pair GEMM of
//                           Gram mode (columns through R0's token list), or
//                           an int32-tile GEMM against R0 (kept sets of more
//                           than kCosMaxCols tokens; smaller ones take the
//                           maxima from the GEMM's cosine-max epilogue).
//   select_candidates_kernel  the diversity stage's candidates: the free
//                           tokens with the smallest of those maxima (after
//                           merging the epilogue's per-column-tile maxima).
// Every ranking orders by (score, lower token index first).
#include <cuda_fp16.h>

#include <algorithm>

#include "p4q.h"
#include "p4q_device.cuh"
#include "p4q_internal.h"
#include "p4q_rank.cuh"

namespace p4q {
namespace {

size_t align256(size_t x) { return (x + 255) & ~static_cast<size_t>(255); }

// Upper bound on the stages-1/2 block: one thread per kPer tokens (N <= 4096).
constexpr int kSelThreads = 1024;

struct RankScratch {
  unsigned int hist[256];
  unsigned int wsum[32];
  int digit, above;
};

// Stages 1 and 2 of Eq. 4 for image blockIdx.x, on blockDim.x = ceil(N / 4)
// rounded up to a warp: query relevance (one ranking per concept, quota
// floor(Kq / J) + (j < Kq % J), each concept keeps its best tokens not yet
// kept), then visual saliency (the best Ks of A_cls among the rest). The kept
// set R0 goes out as bits (token t: bit t % 32 of word t / 32 of the image's
// row of kept12), as the ascending list r0tok [B, R0] (R0 = Kq + Ks), and as
// idx when there is no diversity stage.
template <int kMaxThreads>
__global__ void __launch_bounds__(kMaxThreads, 1)
    select_stages12_kernel(const float* __restrict__ qdots, int qp, const int32_t* __restrict__ qnorm,
                           const int32_t* __restrict__ vnorm, const float* __restrict__ A_cls, int N, int J, int Kq,
                           int Ks, int Kd, uint32_t* __restrict__ kept12, int32_t* __restrict__ r0tok,
                           int32_t* __restrict__ idx) {
  pdl_wait();
  pdl_launch_dependents();
  __shared__ RankScratch s;
  const int b = blockIdx.x, nt = blockDim.x;
  const int base = kPer * threadIdx.x;
  bool kept[kPer];
#pragma unroll
  for (int e = 0; e < kPer; ++e) kept[e] = false;
  uint32_t key[kPer];
  int nv[kPer];  // squared code norms of the thread's tokens
#pragma unroll
  for (int e = 0; e < kPer; ++e) nv[e] = (Kq > 0 && base + e < N) ? vnorm[static_cast<size_t>(b) * N + base + e] : 0;
  for (int j = 0; j < J && Kq > 0; ++j) {
    const int quota = Kq / J + (j < Kq % J ? 1 : 0);
    const int nq = qnorm[b * J + j];
    // Eq. 4 query cosine of each token with concept j, from the exact dot products
#pragma unroll
    for (int e = 0; e < kPer; ++e) {
      const size_t t = static_cast<size_t>(b) * N + base + e;
      key[e] = (base + e < N) ? float_order_key(code_cosine(static_cast<int>(qdots[t * qp + j]), nq, nv[e])) : 0u;
    }
    block_take_top(key, kept, base, N, quota, nt, s);
  }
  if (Ks > 0) {
    const float* a = A_cls + static_cast<size_t>(b) * N;
#pragma unroll
    for (int e = 0; e < kPer; ++e) key[e] = (base + e < N) ? float_order_key(a[base + e]) : 0u;
    block_take_top(key, kept, base, N, Ks, nt, s);
  }
  // kept bits: the four tokens of a thread share a word (kPer divides 32)
  uint32_t bits = 0;
#pragma unroll
  for (int e = 0; e < kPer; ++e) bits |= (base + e < N && kept[e]) ? 1u << ((base + e) & 31) : 0u;
  const unsigned word_peers = 0xFFu << (8 * ((threadIdx.x & 31) >> 3));  // the 8 lanes of one 32-token word
  bits = __reduce_or_sync(word_peers, bits);
  const int words = (N + 31) / 32;
  if ((threadIdx.x & 7) == 0 && base / 32 < words) kept12[static_cast<size_t>(b) * words + base / 32] = bits;
  int cnt = 0;
#pragma unroll
  for (int e = 0; e < kPer; ++e) cnt += (base + e < N && kept[e]) ? 1 : 0;
  int total;
  int pos = block_exclusive_scan(cnt, &total, nt, s);
  const int R0 = Kq + Ks;
#pragma unroll
  for (int e = 0; e < kPer; ++e) {
    if (base + e < N && kept[e] && pos < R0) {
      r0tok[static_cast<size_t>(b) * R0 + pos] = base + e;
      if (Kd == 0) idx[static_cast<size_t>(b) * R0 + pos] = base + e;
      ++pos;
    }
  }
}

// Candidates of the diversity stage for image blockIdx.x: the C free tokens
// (not in R0) with the smallest (m, token) pairs, m their largest cosine to
// R0, as an ascending list cand [B, C]. Greedy picks and pool entries are
// taken among the smallest pairs and pairs only grow, so the stage usually
// needs the cosines of candidates only (the GEMM over them); it checks, per
// pool phase, that it does. Same layout and radix select as stages 1-2.
template <int kMaxThreads>
__global__ void __launch_bounds__(kMaxThreads, 1)
    select_candidates_kernel(float* __restrict__ m, const float* __restrict__ mpart, int parts,
                             const uint32_t* __restrict__ kept12, int N, int R0, int C, int32_t* __restrict__ cand) {
  pdl_wait();
  pdl_launch_dependents();
  if (mpart != nullptr) {
    // m = the largest of the per-column-tile maxima (stage 3 reads m too)
    const size_t part = static_cast<size_t>(gridDim.x) * N;
    for (int i = threadIdx.x; i < N; i += blockDim.x) {
      const size_t t = static_cast<size_t>(blockIdx.x) * N + i;
      float v = mpart[t];
      for (int k = 1; k < parts; ++k) v = fmaxf(v, mpart[k * part + t]);
      m[t] = v;
    }
    __syncthreads();
  }
  __shared__ RankScratch s;
  const int b = blockIdx.x, nt = blockDim.x;
  const int base = kPer * threadIdx.x;
  const int words = (N + 31) / 32;
  bool taken[kPer];
  uint32_t key[kPer];
#pragma unroll
  for (int e = 0; e < kPer; ++e) {
    const int i = base + e;
    taken[e] = i < N && ((kept12[static_cast<size_t>(b) * words + (i >> 5)] >> (i & 31)) & 1u);
    // the smallest pairs as the largest keys; m = -inf (R0 empty) ranks every token equal
    key[e] = (i < N) ? ~float_order_key(R0 > 0 ? m[static_cast<size_t>(b) * N + i] : -INFINITY) : 0u;
  }
  bool in_r0[kPer];
#pragma unroll
  for (int e = 0; e < kPer; ++e) in_r0[e] = taken[e];
  block_take_top(key, taken, base, N, C, nt, s);
  int cnt = 0;
#pragma unroll
  for (int e = 0; e < kPer; ++e) cnt += (base + e < N && taken[e] && !in_r0[e]) ? 1 : 0;
  int total;
  int pos = block_exclusive_scan(cnt, &total, nt, s);
#pragma unroll
  for (int e = 0; e < kPer; ++e)
    if (base + e < N && taken[e] && !in_r0[e] && pos < C) cand[static_cast<size_t>(b) * C + pos++] = base + e;
}

// ru[b, j] = vu[b, tok[b, j]] (d bytes), with its row sum and squared norm,
// for R listed tokens per image (the kept set R0, or the candidates of the
// diversity stage): one warp per row, 16-byte chunks.
__global__ void __launch_bounds__(256) gather_rows_kernel(const uint8_t* __restrict__ vu,
                                                          const int32_t* __restrict__ vsum,
                                                          const int32_t* __restrict__ vnorm,
                                                          const int32_t* __restrict__ tok, int B, int N, int d, int R,
                                                          uint8_t* __restrict__ ru, int32_t* __restrict__ rsum,
                                                          int32_t* __restrict__ rnorm) {
  pdl_wait();
  pdl_launch_dependents();
  const int lane = threadIdx.x & 31;
  const int rows = B * R;
  const int nwarps = gridDim.x * (blockDim.x >> 5);
  const int chunks = d >> 4;
  for (int r = blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5); r < rows; r += nwarps) {
    const int b = r / R;
    const size_t src = static_cast<size_t>(b) * N + tok[r];
    const uint4* s = reinterpret_cast<const uint4*>(vu + src * d);
    uint4* t = reinterpret_cast<uint4*>(ru + static_cast<size_t>(r) * d);
    for (int c = lane; c < chunks; c += 32) t[c] = ldg_stream16(s + c);
    if (lane == 0) {
      rsum[r] = vsum[src];
      rnorm[r] = vnorm[src];
    }
  }
}

// m[b, i] = max over j < R0 of cos(token i, R0 token j) from the exact dot
// products (integers held exactly as fp32): one warp per token row, a CTA
// takes kCosmaxRows rows of one image and stages its R0 norms and their
// reciprocal square roots in shared memory. The largest approximate cosine
// first (dot * rsqrtf(na) * rsqrtf(nb): within 1e-6 of the exact cosine, far
// inside kCosMargin), then the exact cosine of the columns within kCosMargin
// of it, so the maximum is exactly code_cosine's.
constexpr int kCosmaxRows = 8;  // one row per warp: many warps in flight

// cols == nullptr: column j of a row is R0 token j (the R0 GEMM's output,
// norms r0norm); else the row holds every token (the Gram mode's cdots) and
// column j is token cols[b, j] (norms from vnorm).
__global__ void __launch_bounds__(256) r0_cosmax_kernel(const float* __restrict__ dots, int pitch,
                                                        const int32_t* __restrict__ vnorm,
                                                        const int32_t* __restrict__ r0norm,
                                                        const int32_t* __restrict__ cols, int N, int R0,
                                                        float* __restrict__ m) {
  extern __shared__ int32_t nr[];  // [R0] squared norms of the image's kept tokens, [R0] their rsqrtf, [R0] columns
  float* rr = reinterpret_cast<float*>(nr + R0);
  int32_t* cj = nr + 2 * R0;
  pdl_wait();
  pdl_launch_dependents();
  const int b = blockIdx.y, lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  for (int j = threadIdx.x; j < R0; j += blockDim.x) {
    const int c = cols ? cols[static_cast<size_t>(b) * R0 + j] : j;
    const int v = cols ? vnorm[static_cast<size_t>(b) * N + c] : r0norm[static_cast<size_t>(b) * R0 + j];
    nr[j] = v;
    rr[j] = v > 0 ? rsqrtf(static_cast<float>(v)) : 0.0f;
    cj[j] = c;
  }
  __syncthreads();
  for (int i = blockIdx.x * kCosmaxRows + warp; i < min(N, (blockIdx.x + 1) * kCosmaxRows); i += blockDim.x / 32) {
    const size_t row = static_cast<size_t>(b) * N + i;
    const float* dr = dots + row * pitch;
    const int na = vnorm[row];
    const float ra = na > 0 ? rsqrtf(static_cast<float>(na)) : 0.0f;
    float amax = -INFINITY;
#pragma unroll 4
    for (int j = lane; j < R0; j += 32) amax = fmaxf(amax, __ldg(dr + cj[j]) * ra * rr[j]);
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) amax = fmaxf(amax, __shfl_xor_sync(0xFFFFFFFFu, amax, o));
    float emax = -INFINITY;
#pragma unroll 4
    for (int j = lane; j < R0; j += 32) {
      const float dot = __ldg(dr + cj[j]);
      if (dot * ra * rr[j] >= amax - kCosMargin) emax = fmaxf(emax, code_cosine(static_cast<int>(dot), na, nr[j]));
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) emax = fmaxf(emax, __shfl_xor_sync(0xFFFFFFFFu, emax, o));
    if (lane == 0) m[row] = emax;
  }
}

// ---------------------------------------------------------------- Top-K replacement ratio
// App. A, Eq. 9: per sample, the Top-K sets of two score rows over the same N
// tokens (ties to the lower index, the selector's radix select) and the size
// of their intersection; rho = 1 - |T_ref & T_alt| / K. One CTA per sample,
// token i = kPer * threadIdx.x + e.
// Order key of a score with -0 and +0 equal (they tie, and the lower index wins).
__device__ __forceinline__ uint32_t score_key(float v) { return float_order_key(v == 0.0f ? 0.0f : v); }

struct TopkScratch {
  unsigned int hist[256];
  unsigned int wsum[32];
  int digit, above;
};

__global__ void __launch_bounds__(kSelThreads)
    topk_replacement_kernel(const float* __restrict__ s_ref, const float* __restrict__ s_alt, int N, int K,
                            int32_t* __restrict__ inter, float* __restrict__ rho) {
  pdl_wait();
  pdl_launch_dependents();
  __shared__ TopkScratch s;
  const int b = blockIdx.x, nt = blockDim.x, base = kPer * threadIdx.x;
  uint32_t key[kPer];
  bool in_ref[kPer], in_alt[kPer];
#pragma unroll
  for (int e = 0; e < kPer; ++e) {
    key[e] = base + e < N ? score_key(s_ref[static_cast<size_t>(b) * N + base + e]) : 0u;
    in_ref[e] = false;
    in_alt[e] = false;
  }
  block_take_top(key, in_ref, base, N, K, nt, s);
#pragma unroll
  for (int e = 0; e < kPer; ++e)
    key[e] = base + e < N ? score_key(s_alt[static_cast<size_t>(b) * N + base + e]) : 0u;
  block_take_top(key, in_alt, base, N, K, nt, s);
  int c = 0;
#pragma unroll
  for (int e = 0; e < kPer; ++e) c += (in_ref[e] && in_alt[e]) ? 1 : 0;
  int total;
  block_exclusive_scan(c, &total, nt, s);
  if (threadIdx.x == 0) {
    inter[b] = total;
    rho[b] = __fsub_rn(1.0f, __fdiv_rn(static_cast<float>(total), static_cast<float>(K)));
  }
}

}  // namespace

cudaError_t launch_topk_replacement(const float* s_ref, const float* s_alt, int B, int N, int K, int32_t* inter,
                                    float* rho, cudaStream_t stream) {
  if (B <= 0) return cudaSuccess;
  const int nt = ((N + kPer - 1) / kPer + 31) / 32 * 32;
  return launch_pdl(topk_replacement_kernel, dim3(B), dim3(nt), 0, stream, s_ref, s_alt, N, K, inter, rho);
}

// Tile width (B rows, a multiple of 32 up to 256) of the GEMM of every token
// with R0: the fewest column tiles, split evenly.
int r0_tile_n(int R0) {
  const int nt = (R0 + 255) / 256;
  const int per = (R0 + nt - 1) / nt;
  return (per + 31) / 32 * 32;
}

bool select_gram_mode(int N, int Kd) { return Kd > 0 && N <= kGramMaxTokens; }

int select_candidates(int N, int R0, int Kd) {
  if (Kd <= 0) return 0;
  if (select_gram_mode(N, Kd)) return N;
  const int want = std::min((Kd + kCandExtra + 31) / 32 * 32, kCandMax);
  return std::min(N - R0, want);
}

size_t select_workspace_layout(int B, int N, int d, int J, int R0, int C, bool gram, SelectWorkspace* ws,
                               void* base) {
  const size_t BN = static_cast<size_t>(B) * N, BJ = static_cast<size_t>(B) * J;
  const bool r0gemm = !gram && C > 0;  // R0's own GEMM (not in Gram mode, nor without a diversity stage)
  const size_t BR = r0gemm ? static_cast<size_t>(B) * R0 : 0;
  const size_t BC = gram ? 0 : static_cast<size_t>(B) * C;   // gathered candidates (not in Gram mode)
  const int cp = (C + 3) & ~3;
  size_t off = 0;
  auto take = [&](size_t bytes) {
    const size_t o = off;
    off += align256(bytes);
    return o;
  };
  const int tn = R0 > 0 ? r0_tile_n(R0) : 32;
  const int dp = (R0 + 3) & ~3;
  const size_t o_vs = take(BN * 4), o_vn = take(BN * 4);
  const size_t o_qc = take(BJ * (d / 2)), o_qs = take(BJ * 4), o_qn = take(BJ * 4);
  const size_t o_qu = take(BJ * d), o_qsum = take(BJ * 4);
  const int qp = (J + 3) & ~3;
  const size_t o_sc = take(BN * qp * 4);
  const size_t o_vu = take(BN * d), o_vsum = take(BN * 4);
  const size_t o_k12 = take(static_cast<size_t>(B) * ((N + 31) / 32) * 4);
  const size_t o_r0t = take(static_cast<size_t>(B) * R0 * 4);
  const size_t o_r0u = take(BR * d), o_r0s = take(BR * 4), o_r0n = take(BR * 4);
  const bool rowpass = r0gemm && R0 > kCosMaxCols;  // int32 tiles and a row pass
  const int parts = (r0gemm && !rowpass && R0 > 0) ? (R0 + tn - 1) / tn : 0;
  const size_t o_dot = take(rowpass ? BN * dp * 4 : 0), o_m = take(BN * 4);
  const size_t o_mp = take(parts > 1 ? parts * BN * 4 : 0);
  const size_t o_ct = take(BC * 4), o_cu = take(BC * d), o_cs = take(BC * 4), o_cn = take(BC * 4);
  const size_t o_cd = take(static_cast<size_t>(B) * C * cp * 4);
  if (ws && base) {
    uint8_t* p = static_cast<uint8_t*>(base);
    ws->vscale = reinterpret_cast<float*>(p + o_vs);
    ws->vnorm = reinterpret_cast<int32_t*>(p + o_vn);
    ws->qcodes = p + o_qc;
    ws->qscale = reinterpret_cast<float*>(p + o_qs);
    ws->qnorm = reinterpret_cast<int32_t*>(p + o_qn);
    ws->qu = p + o_qu;
    ws->qsum = reinterpret_cast<int32_t*>(p + o_qsum);
    ws->qdots = reinterpret_cast<float*>(p + o_sc);
    ws->q_pitch = qp;
    ws->vu = p + o_vu;
    ws->vsum = reinterpret_cast<int32_t*>(p + o_vsum);
    ws->kept12 = reinterpret_cast<uint32_t*>(p + o_k12);
    ws->r0tok = reinterpret_cast<int32_t*>(p + o_r0t);
    ws->r0u = p + o_r0u;
    ws->r0sum = reinterpret_cast<int32_t*>(p + o_r0s);
    ws->r0norm = reinterpret_cast<int32_t*>(p + o_r0n);
    ws->dots = reinterpret_cast<float*>(p + o_dot);
    ws->mpart = reinterpret_cast<float*>(p + o_mp);
    ws->r0_parts = parts;
    ws->dot_pitch = dp;
    ws->r0_tile_n = tn;
    ws->m = reinterpret_cast<float*>(p + o_m);
    ws->C = C;
    ws->cand = reinterpret_cast<int32_t*>(p + o_ct);
    ws->candu = p + o_cu;
    ws->candsum = reinterpret_cast<int32_t*>(p + o_cs);
    ws->candnorm = reinterpret_cast<int32_t*>(p + o_cn);
    ws->cdots = reinterpret_cast<float*>(p + o_cd);
    ws->cpitch = cp;
    ws->gram = gram;
  }
  return off;
}

cudaError_t launch_select_stages12(const SelectPlan& p, const SelectWorkspace& ws, const float* A_cls, int32_t* idx,
                                   cudaStream_t stream) {
  const int nt = ((p.N + kPer - 1) / kPer + 31) / 32 * 32;
  auto args = [&](auto kern) {
    return launch_pdl(kern, dim3(p.B), dim3(nt), 0, stream, ws.qdots, ws.q_pitch, ws.qnorm, ws.vnorm, A_cls, p.N,
                      p.J, p.Kq, p.Ks, p.Kd, ws.kept12, ws.r0tok, idx);
  };
  if (nt <= 512) return args(select_stages12_kernel<512>);
  if (nt <= 768) return args(select_stages12_kernel<768>);
  return args(select_stages12_kernel<kSelThreads>);
}

cudaError_t launch_query_dots(const SelectPlan& p, const SelectWorkspace& ws, cudaStream_t stream) {
  GemmArgs g;
  g.M = p.N;  // A rows: the image's tokens
  g.N = p.J;  // B rows: its concepts (one 32-column tile)
  g.K = p.d;
  g.batch = p.B;
  g.out = GemmOut::kS32;
  g.D = ws.qdots;
  g.d_pitch = ws.q_pitch;
  g.tile_n = 32;
  g.f32_out = true;
  return launch_gemm8(g, ws.vu, ws.vsum, ws.qu, ws.qsum, stream);
}

cudaError_t launch_r0_cosmax(const SelectPlan& p, const SelectWorkspace& ws, cudaStream_t stream) {
  const int R0 = p.Kq + p.Ks;
  if (R0 == 0) return cudaSuccess;
  GemmArgs g;
  g.M = p.N;  // A rows: the image's tokens
  g.N = R0;   // B rows: its kept set
  g.K = p.d;
  g.batch = p.B;
  g.tile_n = ws.r0_tile_n;
  if (R0 <= kCosMaxCols) {
    // each token's largest cosine per column tile straight from the accumulators
    g.out = GemmOut::kCos;
    g.D = ws.r0_parts > 1 ? ws.mpart : ws.m;
    g.norm_a = ws.vnorm;
    g.norm_b = ws.r0norm;
    return launch_gemm8(g, ws.vu, ws.vsum, ws.r0u, ws.r0sum, stream);
  }
  g.out = GemmOut::kS32;
  g.D = ws.dots;
  g.d_pitch = ws.dot_pitch;
  g.f32_out = true;
  cudaError_t e = launch_gemm8(g, ws.vu, ws.vsum, ws.r0u, ws.r0sum, stream);
  if (e != cudaSuccess) return e;
  const dim3 grid((p.N + kCosmaxRows - 1) / kCosmaxRows, p.B);
  return launch_pdl(r0_cosmax_kernel, grid, dim3(256), static_cast<size_t>(R0) * 12, stream, ws.dots,
                    ws.dot_pitch, ws.vnorm, ws.r0norm, static_cast<const int32_t*>(nullptr), p.N, R0, ws.m);
}

cudaError_t launch_gram(const SelectPlan& p, const SelectWorkspace& ws, cudaStream_t stream) {
  GemmArgs g;  // every token against every token of its image
  g.M = p.N;
  g.N = p.N;
  g.K = p.d;
  g.batch = p.B;
  g.out = GemmOut::kS32;
  g.D = ws.cdots;
  g.d_pitch = ws.cpitch;
  g.f32_out = true;
  return launch_gemm8(g, ws.vu, ws.vsum, ws.vu, ws.vsum, stream);
}

cudaError_t launch_gram_cosmax(const SelectPlan& p, const SelectWorkspace& ws, cudaStream_t stream) {
  const int R0 = p.Kq + p.Ks;
  if (R0 == 0) return cudaSuccess;
  const dim3 grid((p.N + kCosmaxRows - 1) / kCosmaxRows, p.B);
  return launch_pdl(r0_cosmax_kernel, grid, dim3(256), static_cast<size_t>(R0) * 12, stream, ws.cdots, ws.cpitch,
                    ws.vnorm, static_cast<const int32_t*>(nullptr), static_cast<const int32_t*>(ws.r0tok), p.N, R0,
                    ws.m);
}

cudaError_t launch_candidates(const SelectPlan& p, const SelectWorkspace& ws, cudaStream_t stream) {
  const int C = ws.C;
  if (C <= 0) return cudaSuccess;
  const int R0 = p.Kq + p.Ks;
  const int nt = ((p.N + kPer - 1) / kPer + 31) / 32 * 32;
  auto go = [&](auto kern) {
    return launch_pdl(kern, dim3(p.B), dim3(nt), 0, stream, ws.m, ws.r0_parts > 1 ? ws.mpart : nullptr,
                      ws.r0_parts, ws.kept12, p.N, R0, C, ws.cand);
  };
  cudaError_t e = nt <= 512 ? go(select_candidates_kernel<512>)
                            : (nt <= 768 ? go(select_candidates_kernel<768>) : go(select_candidates_kernel<kSelThreads>));
  if (e != cudaSuccess) return e;
  const int rows = p.B * C;
  const int blocks = std::min((rows + 7) / 8, 4 * num_sms());
  e = launch_pdl(gather_rows_kernel, dim3(blocks), dim3(256), 0, stream, ws.vu, ws.vsum, ws.vnorm, ws.cand, p.B, p.N,
                 p.d, C, ws.candu, ws.candsum, ws.candnorm);
  if (e != cudaSuccess) return e;
  GemmArgs g;  // every candidate against every candidate of its image
  g.M = C;
  g.N = C;
  g.K = p.d;
  g.batch = p.B;
  g.out = GemmOut::kS32;
  g.D = ws.cdots;
  g.d_pitch = ws.cpitch;
  g.f32_out = true;
  return launch_gemm8(g, ws.candu, ws.candsum, ws.candu, ws.candsum, stream);
}

cudaError_t launch_gather_r0(const SelectPlan& p, const SelectWorkspace& ws, cudaStream_t stream) {
  const int R0 = p.Kq + p.Ks;
  const int rows = p.B * R0;
  if (rows == 0) return cudaSuccess;
  const int blocks = std::min((rows + 7) / 8, 4 * num_sms());
  return launch_pdl(gather_rows_kernel, dim3(blocks), dim3(256), 0, stream, ws.vu, ws.vsum, ws.vnorm, ws.r0tok, p.B,
                    p.N, p.d, R0, ws.r0u, ws.r0sum, ws.r0norm);
}

}  // namespace p4q
