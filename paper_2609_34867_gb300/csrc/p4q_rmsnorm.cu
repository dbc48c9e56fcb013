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
// Kernel: one CTA of 512 threads per row; each thread keeps its chunks of 8
// values in registers, adds their squares into a 128-bit integer, the block
// sums those (warp shuffles, then every thread adds the warp sums in warp
// order), every thread forms r, then y, the row's abs-max (a second block
// reduction) and the codes, written packed and, optionally, expanded one byte
// per code (u = code + 8, the GEMM's order) with their row sum.
#include <cuda_fp16.h>

#include "p4q.h"
#include "p4q_device.cuh"
#include "p4q_internal.h"

namespace p4q {
namespace {

constexpr int kRnThreads = 512;
constexpr int kRnWarps = kRnThreads / 32;
constexpr int kRnMaxChunks = P4Q_MAX_ROW / 8 / kRnThreads;  // chunks of 8 values per thread, at most

__device__ __forceinline__ float pow2f(int k) { return __int_as_float((k + 127) << 23); }

// (hi:lo) += x^2 in units of 2^-48 for the fp16 value with bits b (finite):
// |x| = sig * 2^(e - 25) for a normal value (sig = 1024 + f), f * 2^-24 for a
// subnormal one, so x^2 = sig^2 << 2 (e - 1) units, below 2^80.
__device__ __forceinline__ void add_square(uint32_t b, uint64_t& lo, uint64_t& hi) {
  const uint32_t e = (b >> 10) & 0x1Fu, f = b & 0x3FFu;
  const uint32_t sig = e ? (f | 0x400u) : f;
  const uint32_t sh = e ? 2u * (e - 1u) : 0u;          // <= 58
  const uint64_t v = static_cast<uint64_t>(sig * sig);  // < 2^22
  const uint64_t vl = v << sh;
  const uint64_t vh = sh > 42u ? (v >> (64u - sh)) : 0ull;
  lo += vl;
  hi += vh + (lo < vl ? 1ull : 0ull);
}

__device__ __forceinline__ void add128(uint64_t& lo, uint64_t& hi, uint64_t lo2, uint64_t hi2) {
  lo += lo2;
  hi += hi2 + (lo < lo2 ? 1ull : 0ull);
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

template <int MAXC, bool EXPANDED>
__global__ void __launch_bounds__(kRnThreads)
    rmsnorm_quant_kernel(const __half* __restrict__ X, long long ldx, const __half* __restrict__ w, float eps, int K,
                         uint8_t* __restrict__ Xq, float* __restrict__ s_a, uint8_t* __restrict__ Xu,
                         int32_t* __restrict__ sum_xu) {
  pdl_wait();
  pdl_launch_dependents();
  __shared__ unsigned long long slo[kRnWarps], shi[kRnWarps];
  __shared__ float wmax[kRnWarps];
  __shared__ int wsum[kRnWarps];
  const int row = blockIdx.x, t = threadIdx.x, lane = t & 31, warp = t >> 5;
  const int nch = K >> 3;
  const uint4* x4 = reinterpret_cast<const uint4*>(X + static_cast<size_t>(row) * ldx);
  const uint4* w4 = reinterpret_cast<const uint4*>(w);
  uint4 xv[MAXC];
#pragma unroll
  for (int j = 0; j < MAXC; ++j) {
    const int c = t + j * kRnThreads;
    xv[j] = c < nch ? __ldg(x4 + c) : make_uint4(0u, 0u, 0u, 0u);
  }
  // exact sum of squares
  uint64_t lo = 0, hi = 0;
#pragma unroll
  for (int j = 0; j < MAXC; ++j) {
    const uint32_t xw[4] = {xv[j].x, xv[j].y, xv[j].z, xv[j].w};
#pragma unroll
    for (int e = 0; e < 4; ++e) {
      add_square(xw[e] & 0xFFFFu, lo, hi);
      add_square(xw[e] >> 16, lo, hi);
    }
  }
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
  for (int v = 1; v < kRnWarps; ++v) add128(lo, hi, slo[v], shi[v]);
  const float ms = __fdiv_rn(sum_to_f32(lo, hi), static_cast<float>(K));
  const float den = __fadd_rn(ms, eps);
  const float r = den == 0.0f ? 0.0f : __frcp_rn(__fsqrt_rn(den));
  // y = fp16(fp16(x * r) * w), kept as fp32 values
  float y[MAXC][8];
  float m = 0.0f;
#pragma unroll
  for (int j = 0; j < MAXC; ++j) {
    const int c = t + j * kRnThreads;
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
  for (int v = 0; v < kRnWarps; ++v) a = fmaxf(a, wmax[v]);
  const float s = __fdiv_rn(a, 7.0f);
  const float inv = (a != 0.0f) ? __frcp_rn(s) : 0.0f;
  uint32_t* q4 = reinterpret_cast<uint32_t*>(Xq + static_cast<size_t>(row) * (K >> 1));
  uint2* up2 = EXPANDED ? reinterpret_cast<uint2*>(Xu + static_cast<size_t>(row) * K) : nullptr;
  uint32_t su = 0;
#pragma unroll
  for (int j = 0; j < MAXC; ++j) {
    const int c = t + j * kRnThreads;
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
      for (int v = 0; v < kRnWarps; ++v) tot += wsum[v];
      sum_xu[row] = tot;
    }
  }
}

template <int MAXC>
cudaError_t launch_c(const __half* X, long long ldx, const __half* w, float eps, int M, int K, uint8_t* Xq, float* s_a,
                     uint8_t* Xu, int32_t* sum_xu, cudaStream_t stream) {
  if (Xu)
    return launch_pdl(rmsnorm_quant_kernel<MAXC, true>, dim3(M), dim3(kRnThreads), 0, stream, X, ldx, w, eps, K, Xq,
                      s_a, Xu, sum_xu);
  return launch_pdl(rmsnorm_quant_kernel<MAXC, false>, dim3(M), dim3(kRnThreads), 0, stream, X, ldx, w, eps, K, Xq,
                    s_a, Xu, sum_xu);
}

}  // namespace

cudaError_t launch_rmsnorm_quant(const uint16_t* X16, long long ldx, const uint16_t* w16, float eps, int M, int K,
                                 uint8_t* Xq, float* s_a, uint8_t* Xu, int32_t* sum_xu, cudaStream_t stream) {
  if (M <= 0) return cudaSuccess;
  const __half* X = reinterpret_cast<const __half*>(X16);
  const __half* w = reinterpret_cast<const __half*>(w16);
  const int per = (K / 8 + kRnThreads - 1) / kRnThreads;  // chunks per thread
  if (per <= 1) return launch_c<1>(X, ldx, w, eps, M, K, Xq, s_a, Xu, sum_xu, stream);
  if (per <= 2) return launch_c<2>(X, ldx, w, eps, M, K, Xq, s_a, Xu, sum_xu, stream);
  if (per <= 3) return launch_c<3>(X, ldx, w, eps, M, K, Xq, s_a, Xu, sum_xu, stream);
  return launch_c<kRnMaxChunks>(X, ldx, w, eps, M, K, Xq, s_a, Xu, sum_xu, stream);
}

}  // namespace p4q
