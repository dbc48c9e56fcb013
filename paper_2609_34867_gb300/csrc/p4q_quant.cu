// Per-row symmetric 4-bit quantizer (App. A and App. B.3 of the paper:
// symmetric round-to-nearest, one scale per token or per output channel,
// group size -1, clip ratio 1.0), in fp32:
//   a = max_k |x_k|, s = a / 7 (rounded once), code_k = clamp(rne(x_k / s), -8, 7)
// with x_k / s rounded to fp32 before the round-half-even; a == 0 gives s = 0
// and zero codes. Codes are written packed, two per byte, the even index in
// the low nibble (two's complement).
//
// One CTA of 256 threads quantizes one row; the row is read once from HBM with
// 16-byte loads and kept in registers between the abs-max pass and the
// quantization pass. The same kernel serves the activation quantizer, the
// weight quantizer, the selector's fake-quantized copies (with the squared code
// norm as an extra output) and the fused gather of the pruned sequence.
#include <cuda_fp16.h>

#include "p4q_device.cuh"
#include "p4q_internal.h"

namespace p4q {
namespace {

constexpr int kThreads = 256;
constexpr int kMaxChunks = 8;  // 8 halves per chunk: rows of up to 256 * 8 * 8 = 16384

// Rounded quotient code = round_half_even(fl(x / s)), computed as
// round(x * inv) with inv = fl(1 / s): the two quotients differ by less than
// 2^-19 for |x / s| <= 7 (three roundings of relative size 2^-24), so they
// round to the same integer unless x * inv lies within 2^-17 of a .5
// boundary; there the exact quotient fl(x / s) is computed and rounded.
// |x| <= max|x| bounds the code to [-7, 7], so the clamp to [-8, 7] cannot
// bind. Returns the code as a float and adds its square to n2.
__device__ __forceinline__ float quant_code(float x, float s, float inv, float& n2) {
  const float q = __fmul_rn(x, inv);
  float c = rintf(q);
  if (fabsf(q - c) > 0.5f - 0x1p-17f) c = rintf(__fdiv_rn(x, s));
  n2 = __fmaf_rn(c, c, n2);
  return c;
}

// The low 4 bits of a small integer-valued float's two's complement, via the
// bits of c + 1.5 * 2^23 (exact for |c| < 2^22).
__device__ __forceinline__ uint32_t nibble(float c) { return __float_as_uint(c + 12582912.0f) & 0xFu; }

// Eight fp16 values (one 16-byte chunk) -> eight packed 4-bit codes.
__device__ __forceinline__ uint32_t quant_chunk(const uint4 v, float s, float inv, float& n2) {
  const uint32_t w[4] = {v.x, v.y, v.z, v.w};
  uint32_t packed = 0;
#pragma unroll
  for (int k = 0; k < 4; ++k) {
    const __half2 hv = *reinterpret_cast<const __half2*>(&w[k]);
    const float2 f = __half22float2(hv);
    const uint32_t n0 = nibble(quant_code(f.x, s, inv, n2));
    const uint32_t n1 = nibble(quant_code(f.y, s, inv, n2));
    packed |= (n0 | (n1 << 4)) << (8 * k);
  }
  return packed;
}

__global__ void __launch_bounds__(kThreads) quant_rows_kernel(RowSource src, int L, RowSinks out) {
  const int row = blockIdx.x;
  const uint16_t* srow;
  if (src.idx == nullptr) {
    srow = src.X + static_cast<size_t>(row) * L;
  } else {
    const int per = src.K + src.T;
    const int b = row / per, t = row - b * per;
    if (t < src.K)
      srow = src.X + (static_cast<size_t>(b) * src.N + src.idx[b * src.K + t]) * L;
    else
      srow = src.text + (static_cast<size_t>(b) * src.T + (t - src.K)) * L;
  }
  const int nch = L >> 3;
  const uint4* s4 = reinterpret_cast<const uint4*>(srow);

  uint4 v[kMaxChunks];
  uint32_t m = 0;  // per-halfword max of |x| bit patterns (non-negative fp16 order as integers)
#pragma unroll
  for (int i = 0; i < kMaxChunks; ++i) {
    const int c = threadIdx.x + i * kThreads;
    if (c < nch) {
      v[i] = __ldg(s4 + c);
      m = __vmaxu2(m, v[i].x & 0x7FFF7FFFu);
      m = __vmaxu2(m, v[i].y & 0x7FFF7FFFu);
      m = __vmaxu2(m, v[i].z & 0x7FFF7FFFu);
      m = __vmaxu2(m, v[i].w & 0x7FFF7FFFu);
    }
  }
  uint32_t mm = max(m & 0xFFFFu, m >> 16);
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) mm = max(mm, __shfl_xor_sync(0xFFFFFFFFu, mm, o));
  __shared__ uint32_t red[kThreads / 32];
  __shared__ int red_n[kThreads / 32];
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (lane == 0) red[warp] = mm;
  __syncthreads();
  mm = red[0];
#pragma unroll
  for (int w = 1; w < kThreads / 32; ++w) mm = max(mm, red[w]);
  const float a = __half2float(__ushort_as_half(static_cast<unsigned short>(mm)));
  const float s = __fdiv_rn(a, 7.0f);
  const float inv = (a != 0.0f) ? __frcp_rn(s) : 0.0f;

  float n2 = 0.0f;  // exact: sum of squared codes <= 49 * 16384 < 2^24
  uint32_t* q4 = reinterpret_cast<uint32_t*>(out.codes + static_cast<size_t>(row) * (L >> 1));
#pragma unroll
  for (int i = 0; i < kMaxChunks; ++i) {
    const int c = threadIdx.x + i * kThreads;
    if (c < nch) {
      q4[c] = (a != 0.0f) ? quant_chunk(v[i], s, inv, n2) : 0u;
      if (out.copy) reinterpret_cast<uint4*>(out.copy + static_cast<size_t>(row) * L)[c] = v[i];
    }
  }
  if (out.norm2) {
    const int wn = __reduce_add_sync(0xFFFFFFFFu, static_cast<int>(n2));
    if (lane == 0) red_n[warp] = wn;
    __syncthreads();
    if (threadIdx.x == 0) {
      int t = 0;
#pragma unroll
      for (int w = 0; w < kThreads / 32; ++w) t += red_n[w];
      out.norm2[row] = t;
    }
  }
  if (threadIdx.x == 0) out.scale[row] = (a != 0.0f) ? s : 0.0f;
}

}  // namespace

cudaError_t launch_quant_rows(const RowSource& src, int rows, int L, const RowSinks& out,
                              cudaStream_t stream) {
  if (rows <= 0) return cudaSuccess;
  quant_rows_kernel<<<rows, kThreads, 0, stream>>>(src, L, out);
  return cudaGetLastError();
}

}  // namespace p4q
