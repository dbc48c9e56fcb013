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

__device__ __forceinline__ uint32_t quant_pair(uint32_t h2, float s, int& n2) {
  // h2 holds two fp16 values; returns their two 4-bit codes in bits [0,8).
  const __half2 hv = *reinterpret_cast<const __half2*>(&h2);
  const float x0 = __low2float(hv), x1 = __high2float(hv);
  int c0 = __float2int_rn(__fdiv_rn(x0, s));
  int c1 = __float2int_rn(__fdiv_rn(x1, s));
  c0 = min(max(c0, -8), 7);
  c1 = min(max(c1, -8), 7);
  n2 += c0 * c0 + c1 * c1;
  return (static_cast<uint32_t>(c0) & 0xFu) | ((static_cast<uint32_t>(c1) & 0xFu) << 4);
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

  int n2 = 0;
  uint32_t* q4 = reinterpret_cast<uint32_t*>(out.codes + static_cast<size_t>(row) * (L >> 1));
#pragma unroll
  for (int i = 0; i < kMaxChunks; ++i) {
    const int c = threadIdx.x + i * kThreads;
    if (c < nch) {
      uint32_t packed = 0;
      if (a != 0.0f) {
        packed = quant_pair(v[i].x, s, n2) | (quant_pair(v[i].y, s, n2) << 8) |
                 (quant_pair(v[i].z, s, n2) << 16) | (quant_pair(v[i].w, s, n2) << 24);
      }
      q4[c] = packed;
      if (out.copy) reinterpret_cast<uint4*>(out.copy + static_cast<size_t>(row) * L)[c] = v[i];
    }
  }
  if (out.norm2) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) n2 += __shfl_xor_sync(0xFFFFFFFFu, n2, o);
    if (lane == 0) red_n[warp] = n2;
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
