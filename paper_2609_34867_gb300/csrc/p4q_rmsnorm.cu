// RMSNorm before the quantized linears, fused with the per-token 4-bit
// quantizer of their input (App. A: every linear's input is quantized per
// token; the decoder's input norms feed q/k/v/gate/up):
//   S = sum_k x_k^2 exactly, rounded once to fp32; ms = S / d;
//   r = 1 / sqrt(ms + eps) (0 when ms + eps == 0); t_k = fp16(x_k * r);
//   y_k = fp16(t_k * w_k); then a = max|y|, s = a / 7,
//   code = clamp(round_half_even(y / s), -8, 7).
// Every fp16 value is an integer multiple of 2^-24, so its square is an
// integer count of 2^-48 below 2^80 and the row's sum fits 128 bits: the sum
// is exact whatever the order of the additions, and its one rounding to fp32
// (to nearest, ties to even) is the same on every evaluation. The remaining
// steps are single correctly rounded operations.
//
// The exact sum on the fp32 pipes: a square q = x^2 is exact in fp32 (at most
// 22 significant bits, at least 2^-48). Adding M = 1.5 * 2^(t + 23) to a value
// below 2^(t + 22) rounds it to a multiple of 2^t, and the bits of the sum
// minus those of M are that multiple as an integer; the residual is exact.
// Four such splits (t = 10, -12, -34, -48) write q as
// H1 2^10 + H2 2^-12 + H3 2^-34 + H4 2^-48 with integers |H| <= 2^22; each
// thread adds the bit patterns in four 32-bit words and turns them into one
// 128-bit integer count of 2^-48 at the end.
//
// Kernel: one CTA per row, 128, 256 or 512 threads (so that a thread has at
// most 4 chunks of 8 values, kept in registers); the block sums the 128-bit
// integers (warp shuffles, then every thread adds the warp sums in warp
// order), every thread forms r, then y, the row's abs-max (a second block
// reduction) and the codes, written packed and, optionally, expanded one byte
// per code (u = code + 8, the GEMM's order) with their row sum.
#include <cuda_fp16.h>

#include "p4q.h"
#include "p4q_device.cuh"
#include "p4q_internal.h"

namespace p4q {
namespace {

constexpr int kRnMaxChunks = 4;  // chunks of 8 values per thread, at most

__device__ __forceinline__ float pow2f(int k) { return __int_as_float((k + 127) << 23); }

constexpr float kM1 = 0x1.8p+33f, kM2 = 0x1.8p+11f, kM3 = 0x1.8p-11f, kM4 = 0x1.8p-25f;

// acc[i] += bits of (residual + M_i) for the four splits of q = x^2
__device__ __forceinline__ void add_square(float x, uint32_t (&acc)[4]) {
  const float q = __fmul_rn(x, x);
  const float a1 = __fadd_rn(q, kM1);
  const float r1 = __fsub_rn(q, __fsub_rn(a1, kM1));
  const float a2 = __fadd_rn(r1, kM2);
  const float r2 = __fsub_rn(r1, __fsub_rn(a2, kM2));
  const float a3 = __fadd_rn(r2, kM3);
  const float r3 = __fsub_rn(r2, __fsub_rn(a3, kM3));
  const float a4 = __fadd_rn(r3, kM4);
  acc[0] += __float_as_uint(a1);
  acc[1] += __float_as_uint(a2);
  acc[2] += __float_as_uint(a3);
  acc[3] += __float_as_uint(a4);
}

__device__ __forceinline__ void add128(uint64_t& lo, uint64_t& hi, uint64_t lo2, uint64_t hi2) {
  lo += lo2;
  hi += hi2 + (lo < lo2 ? 1ull : 0ull);
}

__device__ __forceinline__ void add128s(uint64_t& lo, uint64_t& hi, long long v) {
  add128(lo, hi, static_cast<uint64_t>(v), v < 0 ? ~0ull : 0ull);
}

// The thread's sum of squares as a 128-bit count of 2^-48 from the four words
// (each holds n values' bits: n times the bits of M_i plus the sum of the H_i).
__device__ __forceinline__ void acc_to_u128(const uint32_t (&acc)[4], int n, uint64_t& lo, uint64_t& hi) {
  const long long h1 = static_cast<int>(acc[0] - static_cast<uint32_t>(n) * __float_as_uint(kM1));
  const long long h2 = static_cast<int>(acc[1] - static_cast<uint32_t>(n) * __float_as_uint(kM2));
  const long long h3 = static_cast<int>(acc[2] - static_cast<uint32_t>(n) * __float_as_uint(kM3));
  const long long h4 = static_cast<int>(acc[3] - static_cast<uint32_t>(n) * __float_as_uint(kM4));
  lo = static_cast<uint64_t>(h1) << 58;  // h1 >= 0, below 2^27
  hi = static_cast<uint64_t>(h1) >> 6;
  add128s(lo, hi, h2 * (1ll << 36));
  add128s(lo, hi, h3 * (1ll << 14));
  add128s(lo, hi, h4);
}

// fl32(S * 2^-48) for S = hi * 2^64 + lo, hi < 2^30: the top 64 bits of S with
// every lower bit folded into a sticky bit 0 round to 24 bits exactly as S
// does; the power-of-two scaling is exact (the result is a normal number).
__device__ __forceinline__ float sum_to_f32(uint64_t lo, uint64_t hi) {
  if (hi == 0) return __fmul_rn(__ull2float_rn(lo), 0x1p-48f);
  const int lz = __clzll(static_cast<long long>(hi));  // 34 .. 63
  const uint64_t top = (hi << lz) | (lo >> (64 - lz));
  const uint64_t sticky = (lo << lz) != 0ull ? 1ull : 0ull;
  return __fmul_rn(__ull2float_rn(top | sticky), pow2f(16 - lz));
}

template <int THREADS, int MAXC, bool EXPANDED>
__global__ void __launch_bounds__(THREADS)
    rmsnorm_quant_kernel(const __half* __restrict__ X, long long ldx, const __half* __restrict__ w, float eps, int K,
                         uint8_t* __restrict__ Xq, float* __restrict__ s_a, uint8_t* __restrict__ Xu,
                         int32_t* __restrict__ sum_xu) {
  pdl_wait();
  pdl_launch_dependents();
  constexpr int kWarps = THREADS / 32;
  __shared__ unsigned long long slo[kWarps], shi[kWarps];
  __shared__ float wmax[kWarps];
  __shared__ int wsum[kWarps];
  const int row = blockIdx.x, t = threadIdx.x, lane = t & 31, warp = t >> 5;
  const int nch = K >> 3;
  const uint4* x4 = reinterpret_cast<const uint4*>(X + static_cast<size_t>(row) * ldx);
  const uint4* w4 = reinterpret_cast<const uint4*>(w);
  uint4 xv[MAXC];
#pragma unroll
  for (int j = 0; j < MAXC; ++j) {
    const int c = t + j * THREADS;
    xv[j] = c < nch ? __ldg(x4 + c) : make_uint4(0u, 0u, 0u, 0u);
  }
  // exact sum of squares
  uint32_t acc[4] = {0u, 0u, 0u, 0u};
#pragma unroll
  for (int j = 0; j < MAXC; ++j) {
    const uint32_t xw[4] = {xv[j].x, xv[j].y, xv[j].z, xv[j].w};
#pragma unroll
    for (int e = 0; e < 4; ++e) {
      const float2 xf = __half22float2(*reinterpret_cast<const __half2*>(&xw[e]));
      add_square(xf.x, acc);
      add_square(xf.y, acc);
    }
  }
  uint64_t lo, hi;
  acc_to_u128(acc, 8 * MAXC, lo, hi);
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    const uint64_t lo2 = __shfl_xor_sync(0xFFFFFFFFu, lo, o), hi2 = __shfl_xor_sync(0xFFFFFFFFu, hi, o);
    add128(lo, hi, lo2, hi2);
  }
  if (lane == 0) {
    slo[warp] = lo;
    shi[warp] = hi;
  }
  __syncthreads();
  lo = slo[0];
  hi = shi[0];
#pragma unroll
  for (int v = 1; v < kWarps; ++v) add128(lo, hi, slo[v], shi[v]);
  const float ms = __fdiv_rn(sum_to_f32(lo, hi), static_cast<float>(K));
  const float den = __fadd_rn(ms, eps);
  const float r = den == 0.0f ? 0.0f : __frcp_rn(__fsqrt_rn(den));
  // y = fp16(fp16(x * r) * w), kept as fp32 values
  float y[MAXC][8];
  float m = 0.0f;
#pragma unroll
  for (int j = 0; j < MAXC; ++j) {
    const int c = t + j * THREADS;
    const uint4 wv = c < nch ? __ldg(w4 + c) : make_uint4(0u, 0u, 0u, 0u);
    const uint32_t xw[4] = {xv[j].x, xv[j].y, xv[j].z, xv[j].w}, ww[4] = {wv.x, wv.y, wv.z, wv.w};
#pragma unroll
    for (int e = 0; e < 4; ++e) {
      const float2 xf = __half22float2(*reinterpret_cast<const __half2*>(&xw[e]));
      const float2 wf = __half22float2(*reinterpret_cast<const __half2*>(&ww[e]));
      const float t0 = __half2float(__float2half_rn(__fmul_rn(xf.x, r)));
      const float t1 = __half2float(__float2half_rn(__fmul_rn(xf.y, r)));
      y[j][2 * e] = __half2float(__float2half_rn(__fmul_rn(t0, wf.x)));
      y[j][2 * e + 1] = __half2float(__float2half_rn(__fmul_rn(t1, wf.y)));
      m = fmaxf(m, fmaxf(fabsf(y[j][2 * e]), fabsf(y[j][2 * e + 1])));
    }
  }
  m = fmaxf(m, __shfl_xor_sync(0xFFFFFFFFu, m, 16));
  m = fmaxf(m, __shfl_xor_sync(0xFFFFFFFFu, m, 8));
  m = fmaxf(m, __shfl_xor_sync(0xFFFFFFFFu, m, 4));
  m = fmaxf(m, __shfl_xor_sync(0xFFFFFFFFu, m, 2));
  m = fmaxf(m, __shfl_xor_sync(0xFFFFFFFFu, m, 1));
  if (lane == 0) wmax[warp] = m;
  __syncthreads();
  float a = 0.0f;
#pragma unroll
  for (int v = 0; v < kWarps; ++v) a = fmaxf(a, wmax[v]);
  const float s = __fdiv_rn(a, 7.0f);
  const float inv = (a != 0.0f) ? __frcp_rn(s) : 0.0f;
  uint32_t* q4 = reinterpret_cast<uint32_t*>(Xq + static_cast<size_t>(row) * (K >> 1));
  uint2* up2 = EXPANDED ? reinterpret_cast<uint2*>(Xu + static_cast<size_t>(row) * K) : nullptr;
  uint32_t su = 0;
#pragma unroll
  for (int j = 0; j < MAXC; ++j) {
    const int c = t + j * THREADS;
    if (c < nch) {
      // value e of the chunk in bits 4e: byte i holds values 2i (low nibble) and 2i + 1
      uint32_t pw = 0;
      if (a != 0.0f) {
#pragma unroll
        for (int e = 0; e < 8; ++e) pw |= (static_cast<uint32_t>(q4_code(y[j][e], s, inv)) & 0xFu) << (4 * e);
      }
      q4[c] = pw;
      if (EXPANDED) {
        // the even values, then the odd ones, offset by 8 (the GEMM's order)
        const uint32_t eu = (pw & 0x0F0F0F0Fu) ^ 0x08080808u, ou = ((pw >> 4) & 0x0F0F0F0Fu) ^ 0x08080808u;
        up2[c] = make_uint2(eu, ou);
        su = __dp4a(eu + ou, 0x01010101u, su);
      }
    }
  }
  if (t == 0) s_a[row] = (a != 0.0f) ? s : 0.0f;
  if (EXPANDED) {
    const int ws = static_cast<int>(__reduce_add_sync(0xFFFFFFFFu, su));
    if (lane == 0) wsum[warp] = ws;
    __syncthreads();
    if (t == 0) {
      int tot = 0;
#pragma unroll
      for (int v = 0; v < kWarps; ++v) tot += wsum[v];
      sum_xu[row] = tot;
    }
  }
}

template <int THREADS, int MAXC>
cudaError_t launch_c(const __half* X, long long ldx, const __half* w, float eps, int M, int K, uint8_t* Xq, float* s_a,
                     uint8_t* Xu, int32_t* sum_xu, cudaStream_t stream) {
  if (Xu)
    return launch_pdl(rmsnorm_quant_kernel<THREADS, MAXC, true>, dim3(M), dim3(THREADS), 0, stream, X, ldx, w, eps,
                      K, Xq, s_a, Xu, sum_xu);
  return launch_pdl(rmsnorm_quant_kernel<THREADS, MAXC, false>, dim3(M), dim3(THREADS), 0, stream, X, ldx, w, eps, K,
                    Xq, s_a, Xu, sum_xu);
}

template <int THREADS>
cudaError_t launch_t(const __half* X, long long ldx, const __half* w, float eps, int M, int K, uint8_t* Xq, float* s_a,
                     uint8_t* Xu, int32_t* sum_xu, cudaStream_t stream) {
  const int per = (K / 8 + THREADS - 1) / THREADS;  // chunks per thread, at most kRnMaxChunks
  if (per <= 1) return launch_c<THREADS, 1>(X, ldx, w, eps, M, K, Xq, s_a, Xu, sum_xu, stream);
  if (per <= 2) return launch_c<THREADS, 2>(X, ldx, w, eps, M, K, Xq, s_a, Xu, sum_xu, stream);
  if (per <= 3) return launch_c<THREADS, 3>(X, ldx, w, eps, M, K, Xq, s_a, Xu, sum_xu, stream);
  return launch_c<THREADS, kRnMaxChunks>(X, ldx, w, eps, M, K, Xq, s_a, Xu, sum_xu, stream);
}

}  // namespace

cudaError_t launch_rmsnorm_quant(const uint16_t* X16, long long ldx, const uint16_t* w16, float eps, int M, int K,
                                 uint8_t* Xq, float* s_a, uint8_t* Xu, int32_t* sum_xu, cudaStream_t stream) {
  if (M <= 0) return cudaSuccess;
  const __half* X = reinterpret_cast<const __half*>(X16);
  const __half* w = reinterpret_cast<const __half*>(w16);
  static_assert(P4Q_MAX_ROW <= 8 * 512 * kRnMaxChunks, "rows longer than 512 threads x 4 chunks");
  if (K <= 8 * 128 * kRnMaxChunks) return launch_t<128>(X, ldx, w, eps, M, K, Xq, s_a, Xu, sum_xu, stream);
  if (K <= 8 * 256 * kRnMaxChunks) return launch_t<256>(X, ldx, w, eps, M, K, Xq, s_a, Xu, sum_xu, stream);
  return launch_t<512>(X, ldx, w, eps, M, K, Xq, s_a, Xu, sum_xu, stream);
}

}  // namespace p4q
