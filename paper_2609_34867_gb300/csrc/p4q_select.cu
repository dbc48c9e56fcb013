// Quantization-aware visual-token selector (Sec. 3.2, Eq. 4 of the paper).
//
// Inputs are the fake-quantized copies produced by the per-row quantizer:
// packed INT4 codes and the squared code norm of every visual token and every
// concept embedding. The cosine of two fake-quantized rows is evaluated on
// their codes (the positive per-row scales cancel):
//   cos(a, b) = (float)<c_a, c_b> / sqrtf((float)|c_a|^2 * (float)|c_b|^2)
// with every operation rounded to fp32 in that order, and 0 when a norm is 0.
//
// Kernels:
//   query_scores_kernel   one warp per visual token: integer dot products with
//                         the J concept codes (dp4a on the offset codes
//                         u = c + 8, corrected by the code sums), then the
//                         cosine per concept.
//   select_stages_kernel  one 1024-thread CTA per image: stage 1 (per-concept
//                         top quota), stage 2 (CLS-saliency top K_s), stage 3
//                         (greedy max-min diversity on the cosine matrix of
//                         the image, computed beforehand on the tensor cores),
//                         then the kept set in ascending order.
// Every ranking orders by (score, lower token index first).
#include <cuda_fp16.h>

#include "p4q.h"
#include "p4q_device.cuh"
#include "p4q_internal.h"

namespace p4q {
namespace {

__device__ __forceinline__ uint32_t lo_u(uint32_t w) { return (w & 0x0F0F0F0Fu) ^ 0x08080808u; }
__device__ __forceinline__ uint32_t hi_u(uint32_t w) { return ((w >> 4) & 0x0F0F0F0Fu) ^ 0x08080808u; }

__device__ __forceinline__ float code_cosine(int dot, int na, int nb) {
  if (na == 0 || nb == 0) return 0.0f;
  return __fdiv_rn(static_cast<float>(dot), __fsqrt_rn(__fmul_rn(static_cast<float>(na), static_cast<float>(nb))));
}

constexpr int kScoreWarps = 8;

// scores[b, j, i] = cos(concept j of image b, token i of image b)
__global__ void __launch_bounds__(kScoreWarps * 32)
    query_scores_kernel(const uint8_t* __restrict__ vcodes, const int32_t* __restrict__ vnorm,
                        const uint8_t* __restrict__ qcodes, const int32_t* __restrict__ qnorm, int B, int N, int d,
                        int J, float* __restrict__ scores) {
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int tok = blockIdx.x * kScoreWarps + warp;
  if (tok >= B * N) return;
  const int b = tok / N, i = tok - b * N;
  const int words = d >> 3;  // 8 codes per 32-bit word
  const uint32_t* tv = reinterpret_cast<const uint32_t*>(vcodes + static_cast<size_t>(tok) * (d >> 1));
  const uint32_t* tq = reinterpret_cast<const uint32_t*>(qcodes + static_cast<size_t>(b) * J * (d >> 1));
  unsigned int P[P4Q_MAX_CONCEPTS];
  unsigned int SQ[P4Q_MAX_CONCEPTS];
#pragma unroll
  for (int j = 0; j < P4Q_MAX_CONCEPTS; ++j) P[j] = SQ[j] = 0;
  unsigned int SV = 0;
  for (int w = lane; w < words; w += 32) {
    const uint32_t x = __ldg(tv + w);
    const uint32_t xl = lo_u(x), xh = hi_u(x);
    SV = __dp4a(xl + xh, 0x01010101u, SV);
#pragma unroll
    for (int j = 0; j < P4Q_MAX_CONCEPTS; ++j) {
      if (j < J) {
        const uint32_t y = __ldg(tq + static_cast<size_t>(j) * words + w);
        const uint32_t yl = lo_u(y), yh = hi_u(y);
        P[j] = __dp4a(xl, yl, P[j]);
        P[j] = __dp4a(xh, yh, P[j]);
        SQ[j] = __dp4a(yl + yh, 0x01010101u, SQ[j]);
      }
    }
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) SV += __shfl_xor_sync(0xFFFFFFFFu, SV, o);
  const int nv = vnorm[tok];
#pragma unroll
  for (int j = 0; j < P4Q_MAX_CONCEPTS; ++j) {
    if (j < J) {
      unsigned int pj = P[j], sj = SQ[j];
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) {
        pj += __shfl_xor_sync(0xFFFFFFFFu, pj, o);
        sj += __shfl_xor_sync(0xFFFFFFFFu, sj, o);
      }
      if (lane == 0) {
        const int dot = static_cast<int>(pj) - 8 * static_cast<int>(SV) - 8 * static_cast<int>(sj) + 64 * d;
        scores[(static_cast<size_t>(b) * J + j) * N + i] = code_cosine(dot, qnorm[b * J + j], nv);
      }
    }
  }
}

constexpr int kSelThreads = 1024;
constexpr int kPer = 4;  // tokens per thread: token i = kPer * threadIdx.x + e

struct BlockScratch {
  unsigned int hist[256];
  unsigned int wsum[32];
  unsigned long long wmin[2][32];
  int digit, above;
  int list_len;
  int list[P4Q_MAX_TOKENS];
};

// Exclusive prefix sum over the block of per-thread counts (thread order).
__device__ int block_exclusive_scan(int v, int* total, BlockScratch& s) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  int x = v;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const int y = __shfl_up_sync(0xFFFFFFFFu, x, o);
    if (lane >= o) x += y;
  }
  if (lane == 31) s.wsum[warp] = x;
  __syncthreads();
  if (warp == 0) {
    int w = s.wsum[lane];
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int y = __shfl_up_sync(0xFFFFFFFFu, w, o);
      if (lane >= o) w += y;
    }
    s.wsum[lane] = w;  // inclusive
  }
  __syncthreads();
  const int before = (warp ? s.wsum[warp - 1] : 0) + x - v;
  *total = s.wsum[31];
  __syncthreads();
  return before;
}

// Marks as kept the q free tokens with the largest keys (keys are the
// order-preserving images of fp32 scores; ties go to the lower token index).
__device__ void block_take_top(const uint32_t (&key)[kPer], bool (&kept)[kPer], int n_valid_base, int N, int q,
                               BlockScratch& s) {
  if (q <= 0) return;
  uint32_t prefix = 0, mask = 0;
  int need = q;
  for (int pass = 0; pass < 4; ++pass) {
    const int shift = 24 - 8 * pass;
    for (int h = threadIdx.x; h < 256; h += blockDim.x) s.hist[h] = 0;
    __syncthreads();
#pragma unroll
    for (int e = 0; e < kPer; ++e) {
      const int i = n_valid_base + e;
      if (i < N && !kept[e] && (key[e] & mask) == prefix) atomicAdd(&s.hist[(key[e] >> shift) & 255u], 1u);
    }
    __syncthreads();
    if (threadIdx.x < 32) {
      // lane l owns digits [8l, 8l+8); find the digit where the count from the top reaches need
      const int lane = threadIdx.x;
      unsigned int c[8], own = 0;
#pragma unroll
      for (int k = 0; k < 8; ++k) {
        c[k] = s.hist[8 * lane + k];
        own += c[k];
      }
      unsigned int above = 0;  // counts of lanes with higher digits
      unsigned int x = own;
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const unsigned int y = __shfl_down_sync(0xFFFFFFFFu, x, o);
        if (lane + o < 32) x += y;
      }
      above = x - own;  // sum over lanes > lane
      if (above < static_cast<unsigned>(need) && above + own >= static_cast<unsigned>(need)) {
        unsigned int acc = above;
        for (int k = 7; k >= 0; --k) {
          if (acc + c[k] >= static_cast<unsigned>(need)) {
            s.digit = 8 * lane + k;
            s.above = static_cast<int>(acc);
            break;
          }
          acc += c[k];
        }
      }
    }
    __syncthreads();
    need -= s.above;
    prefix |= static_cast<uint32_t>(s.digit) << shift;
    mask |= 255u << shift;
    __syncthreads();
  }
  // keys > prefix are taken; among keys == prefix the first `need` in index order
  int eq = 0;
#pragma unroll
  for (int e = 0; e < kPer; ++e) {
    const int i = n_valid_base + e;
    if (i < N && !kept[e] && key[e] == prefix) ++eq;
  }
  int total;
  int rank = block_exclusive_scan(eq, &total, s);
#pragma unroll
  for (int e = 0; e < kPer; ++e) {
    const int i = n_valid_base + e;
    if (i < N && !kept[e]) {
      if (key[e] > prefix) {
        kept[e] = true;
      } else if (key[e] == prefix) {
        if (rank < need) kept[e] = true;
        ++rank;
      }
    }
  }
  __syncthreads();
}

__global__ void __launch_bounds__(kSelThreads, 1)
    select_stages_kernel(const float* __restrict__ scores, const float* __restrict__ A_cls,
                         const float* __restrict__ gram, int gp, int N, int J, int K, int Kq, int Ks,
                         int Kd, int32_t* __restrict__ idx) {
  extern __shared__ uint8_t smem_raw[];
  BlockScratch& s = *reinterpret_cast<BlockScratch*>(smem_raw);
  const int b = blockIdx.x;
  const int base = kPer * threadIdx.x;
  bool kept[kPer];
#pragma unroll
  for (int e = 0; e < kPer; ++e) kept[e] = false;
  uint32_t key[kPer];

  // Stage 1: query relevance, one ranking per concept, quota floor(Kq/J) + (j < Kq % J).
  for (int j = 0; j < J && Kq > 0; ++j) {
    const int quota = Kq / J + (j < Kq % J ? 1 : 0);
    const float* sc = scores + (static_cast<size_t>(b) * J + j) * N;
#pragma unroll
    for (int e = 0; e < kPer; ++e) key[e] = (base + e < N) ? float_order_key(sc[base + e]) : 0u;
    block_take_top(key, kept, base, N, quota, s);
  }
  // Stage 2: visual saliency on the tokens not kept.
  if (Ks > 0) {
    const float* a = A_cls + static_cast<size_t>(b) * N;
#pragma unroll
    for (int e = 0; e < kPer; ++e) key[e] = (base + e < N) ? float_order_key(a[base + e]) : 0u;
    block_take_top(key, kept, base, N, Ks, s);
  }
  // Stage 3: greedy max-min diversity.
  if (Kd > 0) {
    const float* G = gram + static_cast<size_t>(b) * N * gp;
    // list of the kept set R0
    int cnt = 0;
#pragma unroll
    for (int e = 0; e < kPer; ++e) cnt += (base + e < N && kept[e]) ? 1 : 0;
    int total;
    int pos = block_exclusive_scan(cnt, &total, s);
#pragma unroll
    for (int e = 0; e < kPer; ++e)
      if (base + e < N && kept[e]) s.list[pos++] = base + e;
    __syncthreads();
    float m[kPer];
#pragma unroll
    for (int e = 0; e < kPer; ++e) m[e] = -INFINITY;
    const bool full4 = (base + kPer <= N);  // rows start 16-byte aligned (pitch % 4 == 0)
    for (int r = 0; r < total; ++r) {
      const float* row = G + static_cast<size_t>(s.list[r]) * gp;
      if (full4) {
        const float4 g = *reinterpret_cast<const float4*>(row + base);
        m[0] = fmaxf(m[0], g.x); m[1] = fmaxf(m[1], g.y); m[2] = fmaxf(m[2], g.z); m[3] = fmaxf(m[3], g.w);
      } else {
#pragma unroll
        for (int e = 0; e < kPer; ++e)
          if (base + e < N) m[e] = fmaxf(m[e], row[base + e]);
      }
    }
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    for (int t = 0; t < Kd; ++t) {
      unsigned long long best = ~0ull;
#pragma unroll
      for (int e = 0; e < kPer; ++e) {
        if (base + e < N && !kept[e]) {
          const unsigned long long k =
              (static_cast<unsigned long long>(float_order_key(m[e])) << 32) | static_cast<unsigned>(base + e);
          best = k < best ? k : best;
        }
      }
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) {
        const unsigned long long y = __shfl_xor_sync(0xFFFFFFFFu, best, o);
        best = y < best ? y : best;
      }
      const int slot = t & 1;
      if (lane == 0) s.wmin[slot][warp] = best;
      __syncthreads();
      best = s.wmin[slot][lane];
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) {
        const unsigned long long y = __shfl_xor_sync(0xFFFFFFFFu, best, o);
        best = y < best ? y : best;
      }
      const int pick = static_cast<int>(best & 0xFFFFFFFFull);
      if (pick >= base && pick < base + kPer) kept[pick - base] = true;
      const float* row = G + static_cast<size_t>(pick) * gp;
      if (full4) {
        const float4 g = *reinterpret_cast<const float4*>(row + base);
        m[0] = fmaxf(m[0], g.x); m[1] = fmaxf(m[1], g.y); m[2] = fmaxf(m[2], g.z); m[3] = fmaxf(m[3], g.w);
      } else {
#pragma unroll
        for (int e = 0; e < kPer; ++e)
          if (base + e < N) m[e] = fmaxf(m[e], row[base + e]);
      }
    }
  }
  // Output: the kept set in ascending index order.
  int cnt = 0;
#pragma unroll
  for (int e = 0; e < kPer; ++e) cnt += (base + e < N && kept[e]) ? 1 : 0;
  int total;
  int pos = block_exclusive_scan(cnt, &total, s);
#pragma unroll
  for (int e = 0; e < kPer; ++e)
    if (base + e < N && kept[e] && pos < K) idx[static_cast<size_t>(b) * K + pos++] = base + e;
}

size_t align256(size_t x) { return (x + 255) & ~static_cast<size_t>(255); }

}  // namespace

size_t select_workspace_layout(int B, int N, int d, int J, SelectWorkspace* ws, void* base) {
  const size_t BN = static_cast<size_t>(B) * N, BJ = static_cast<size_t>(B) * J;
  size_t off = 0;
  auto take = [&](size_t bytes) {
    const size_t o = off;
    off += align256(bytes);
    return o;
  };
  const size_t o_vc = take(BN * (d / 2)), o_vs = take(BN * 4), o_vn = take(BN * 4);
  const size_t o_qc = take(BJ * (d / 2)), o_qs = take(BJ * 4), o_qn = take(BJ * 4);
  const int gp = (N + 3) & ~3;
  const size_t o_sc = take(BJ * N * 4), o_g = take(BN * gp * 4);
  if (ws && base) {
    uint8_t* p = static_cast<uint8_t*>(base);
    ws->vcodes = p + o_vc;
    ws->vscale = reinterpret_cast<float*>(p + o_vs);
    ws->vnorm = reinterpret_cast<int32_t*>(p + o_vn);
    ws->qcodes = p + o_qc;
    ws->qscale = reinterpret_cast<float*>(p + o_qs);
    ws->qnorm = reinterpret_cast<int32_t*>(p + o_qn);
    ws->scores = reinterpret_cast<float*>(p + o_sc);
    ws->gram = reinterpret_cast<float*>(p + o_g);
    ws->gram_pitch = gp;
  }
  return off;
}

cudaError_t launch_query_scores(const SelectPlan& p, const SelectWorkspace& ws, cudaStream_t stream) {
  const int toks = p.B * p.N;
  query_scores_kernel<<<(toks + kScoreWarps - 1) / kScoreWarps, kScoreWarps * 32, 0, stream>>>(
      ws.vcodes, ws.vnorm, ws.qcodes, ws.qnorm, p.B, p.N, p.d, p.J, ws.scores);
  return cudaGetLastError();
}

cudaError_t launch_select_stages(const SelectPlan& p, const SelectWorkspace& ws, const float* A_cls, int32_t* idx,
                                 cudaStream_t stream) {
  static bool attr_set = false;
  const int smem = static_cast<int>(sizeof(BlockScratch));
  if (!attr_set) {
    cudaError_t e = cudaFuncSetAttribute(select_stages_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
    if (e != cudaSuccess) return e;
    attr_set = true;
  }
  select_stages_kernel<<<p.B, kSelThreads, smem, stream>>>(ws.scores, A_cls, ws.gram, ws.gram_pitch, p.N, p.J,
                                                           p.K, p.Kq, p.Ks, p.Kd, idx);
  return cudaGetLastError();
}

}  // namespace p4q
