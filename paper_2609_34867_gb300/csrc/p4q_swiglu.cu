// SwiGLU before down_proj, fused with the per-token 4-bit quantizer of
// down_proj's input (App. A: every linear's input is quantized per token):
//   h = silu(gate) * up, silu(g) = g * (1 / (1 + exp32(-g))) (each
//   operation one rounded fp32 step, the reciprocal correctly rounded),
//   then a = max|h|, s = a / 7, code = clamp(round_half_even(h / s), -8, 7).
// exp32 is an own fp32 exponential (Cody-Waite reduction with ln 2 split as
// 355/512 + a low part, degree-7 Taylor polynomial by Horner's rule with fused
// multiply-adds, two exact power-of-two scalings; within 0.9 ulp of e^x; 0
// below -87, inf above 88.72284). The fp32 h is within 2.9 ulp (3.5e-7
// relative: 0.9 ulp from exp32 and four roundings of 2^-24) of the real
// silu(g) * up, the row's abs-max likewise, the scale a / 7 adds one
// rounding and the quotient h / s one more, so h / s is within 8.1e-7
// relative, 5.7e-6 absolute (|h / s| <= 7), of the exact quotient: the codes
// are those of the exact SwiGLU except where that quotient falls within
// 5.7e-6 of a .5 boundary.
//
// Kernel: one CTA of 512 threads per row; each thread holds its chunks of 8
// values of h in registers (computed once), the row's abs-max comes from a
// block reduction, then the codes are written packed and, optionally, expanded
// one byte per code (u = code + 8, the GEMM's order) with their row sum.
#include <cuda_fp16.h>

#include "p4q.h"
#include "p4q_device.cuh"
#include "p4q_internal.h"

namespace p4q {
namespace {

constexpr int kSwThreads = 512;
constexpr int kSwMaxChunks = P4Q_MAX_ROW / 8 / kSwThreads;  // chunks of 8 values per thread, at most

__device__ __forceinline__ float pow2f(int k) { return __int_as_float((k + 127) << 23); }

__device__ __forceinline__ float exp32(float x) {
  if (x > 0x1.62e430p+6f) return __int_as_float(0x7f800000);
  if (x < -87.0f) return 0.0f;
  // n = round_half_even(x * log2 e) by adding 1.5 * 2^23 (|n| <= 128); its
  // bits hold n in the low mantissa bits
  const float nm = __fadd_rn(__fmul_rn(x, 0x1.715476p+0f), 12582912.0f);
  const float n = __fsub_rn(nm, 12582912.0f);
  const int k = __float_as_int(nm) - 0x4B400000;
  float r = __fmaf_rn(-n, 0x1.630000p-1f, x);
  r = __fmaf_rn(-n, -0x1.bd0106p-13f, r);
  float p = 0x1.a01a02p-13f;
  p = __fmaf_rn(p, r, 0x1.6c16c2p-10f);
  p = __fmaf_rn(p, r, 0x1.111112p-7f);
  p = __fmaf_rn(p, r, 0x1.555556p-5f);
  p = __fmaf_rn(p, r, 0x1.555556p-3f);
  p = __fmaf_rn(p, r, 0.5f);
  p = __fmaf_rn(p, r, 1.0f);
  p = __fmaf_rn(p, r, 1.0f);
  // p * 2^n is exact (a normal result): one multiplication, two when 2^n
  // itself overflows (n = 128)
  if (k <= 127) return __fmul_rn(p, pow2f(k));
  return __fmul_rn(__fmul_rn(p, pow2f(64)), pow2f(k - 64));
}

// silu(g) * u = (g * (1 / (1 + exp32(-g)))) * u, four rounded fp32 steps
__device__ __forceinline__ float swiglu(float g, float u) {
  const float sig = __frcp_rn(__fadd_rn(1.0f, exp32(-g)));
  return __fmul_rn(__fmul_rn(g, sig), u);
}

template <int MAXC, bool EXPANDED>
__global__ void __launch_bounds__(kSwThreads)
    swiglu_quant_kernel(const __half* __restrict__ gate, long long ldg, const __half* __restrict__ up, long long ldu,
                        int K, uint8_t* __restrict__ Xq, float* __restrict__ s_a, uint8_t* __restrict__ Xu,
                        int32_t* __restrict__ sum_xu) {
  pdl_wait();
  pdl_launch_dependents();
  __shared__ float wmax[kSwThreads / 32];
  __shared__ int wsum[kSwThreads / 32];
  const int row = blockIdx.x, t = threadIdx.x, lane = t & 31, warp = t >> 5;
  const int nch = K >> 3;
  const uint4* g4 = reinterpret_cast<const uint4*>(gate + static_cast<size_t>(row) * ldg);
  const uint4* u4 = reinterpret_cast<const uint4*>(up + static_cast<size_t>(row) * ldu);
  float h[MAXC][8];
  uint4 gv[MAXC], uv[MAXC];
#pragma unroll
  for (int j = 0; j < MAXC; ++j) {
    const int c = t + j * kSwThreads;
    gv[j] = c < nch ? __ldg(g4 + c) : make_uint4(0u, 0u, 0u, 0u);
    uv[j] = c < nch ? __ldg(u4 + c) : make_uint4(0u, 0u, 0u, 0u);
  }
  float m = 0.0f;
#pragma unroll
  for (int j = 0; j < MAXC; ++j) {
    const uint32_t gw[4] = {gv[j].x, gv[j].y, gv[j].z, gv[j].w}, uw[4] = {uv[j].x, uv[j].y, uv[j].z, uv[j].w};
#pragma unroll
    for (int e = 0; e < 4; ++e) {
      const float2 gf = __half22float2(*reinterpret_cast<const __half2*>(&gw[e]));
      const float2 uf = __half22float2(*reinterpret_cast<const __half2*>(&uw[e]));
      h[j][2 * e] = swiglu(gf.x, uf.x);
      h[j][2 * e + 1] = swiglu(gf.y, uf.y);
      m = fmaxf(m, fmaxf(fabsf(h[j][2 * e]), fabsf(h[j][2 * e + 1])));
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
  for (int w = 0; w < kSwThreads / 32; ++w) a = fmaxf(a, wmax[w]);
  const float s = __fdiv_rn(a, 7.0f);
  const float inv = (a != 0.0f) ? __frcp_rn(s) : 0.0f;
  uint32_t* q4 = reinterpret_cast<uint32_t*>(Xq + static_cast<size_t>(row) * (K >> 1));
  uint2* up2 = EXPANDED ? reinterpret_cast<uint2*>(Xu + static_cast<size_t>(row) * K) : nullptr;
  uint32_t su = 0;
#pragma unroll
  for (int j = 0; j < MAXC; ++j) {
    const int c = t + j * kSwThreads;
    if (c < nch) {
      // value e of the chunk in bits 4e: byte i holds values 2i (low nibble) and 2i + 1
      uint32_t pw = 0;
      if (a != 0.0f) {
#pragma unroll
        for (int e = 0; e < 8; ++e) pw |= (static_cast<uint32_t>(q4_code(h[j][e], s, inv)) & 0xFu) << (4 * e);
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
      for (int w = 0; w < kSwThreads / 32; ++w) tot += wsum[w];
      sum_xu[row] = tot;
    }
  }
}

template <int MAXC>
cudaError_t launch_c(const __half* g, long long ldg, const __half* u, long long ldu, int M, int K, uint8_t* Xq,
                     float* s_a, uint8_t* Xu, int32_t* sum_xu, cudaStream_t stream) {
  if (Xu)
    return launch_pdl(swiglu_quant_kernel<MAXC, true>, dim3(M), dim3(kSwThreads), 0, stream, g, ldg, u, ldu, K, Xq,
                      s_a, Xu, sum_xu);
  return launch_pdl(swiglu_quant_kernel<MAXC, false>, dim3(M), dim3(kSwThreads), 0, stream, g, ldg, u, ldu, K, Xq,
                    s_a, Xu, sum_xu);
}

}  // namespace

cudaError_t launch_swiglu_quant(const uint16_t* gate, long long ldg, const uint16_t* up, long long ldu, int M, int K,
                                uint8_t* Xq, float* s_a, uint8_t* Xu, int32_t* sum_xu, cudaStream_t stream) {
  if (M <= 0) return cudaSuccess;
  const __half* g = reinterpret_cast<const __half*>(gate);
  const __half* u = reinterpret_cast<const __half*>(up);
  const int per = (K / 8 + kSwThreads - 1) / kSwThreads;  // chunks per thread
  if (per <= 1) return launch_c<1>(g, ldg, u, ldu, M, K, Xq, s_a, Xu, sum_xu, stream);
  if (per <= 2) return launch_c<2>(g, ldg, u, ldu, M, K, Xq, s_a, Xu, sum_xu, stream);
  if (per <= 3) return launch_c<3>(g, ldg, u, ldu, M, K, Xq, s_a, Xu, sum_xu, stream);
  return launch_c<kSwMaxChunks>(g, ldg, u, ldu, M, K, Xq, s_a, Xu, sum_xu, stream);
}

}  // namespace p4q
