// Per-row symmetric 4-bit quantizer (App. A and App. B.3 of the paper:
// symmetric round-to-nearest, one scale per token or per output channel,
// group size -1, clip ratio 1.0), in fp32:
//   a = max_k |x_k|, s = a / 7 (rounded once), code_k = clamp(rne(x_k / s), -8, 7)
// with x_k / s rounded to fp32 before the round-half-even; a == 0 gives s = 0
// and zero codes. Codes are written packed, two per byte, the even index in
// the low nibble (two's complement).
//
// A warp (rows up to 5120) or four warps (longer rows) quantize one row; the
// row is read once from HBM with 16-byte loads and kept in registers between
// the abs-max pass and the quantization pass. The same kernel serves the activation quantizer, the
// weight quantizer, the selector's fake-quantized copies (with the squared code
// norm as an extra output) and the fused gather of the pruned sequence.
#include <cuda_fp16.h>

#include "p4q_device.cuh"
#include "p4q_internal.h"

namespace p4q {
namespace {

constexpr int kThreads = 256;

// Codes of eight fp16 values (one 16-byte chunk), packed two per byte.
//
// code = round_half_even(fl(x / s)) is computed as round(x * inv) with
// inv = fl(1 / s): the two quotients differ by less than 2^-19 for |x / s| <= 7
// (three roundings of relative size 2^-24), so they round to the same integer
// unless x * inv lies within 2^-17 of a .5 boundary; a chunk with such a value
// is recomputed with exact quotients fl(x / s). Rounding uses the magic
// constant 1.5 * 2^23: q + 1.5 * 2^23 rounds q to the nearest integer (ties
// to even) and leaves its two's complement in the low mantissa bits, which
// are the packed nibble. |x| <= max|x| bounds the codes to [-7, 7], so the
// clamp to [-8, 7] cannot bind. Squares of the codes are added to n2.
__device__ __forceinline__ uint32_t quant_chunk(const uint4 v, float s, float inv, float2& n2) {
  const float2 inv2 = make_float2(inv, inv);
  const float2 mg = make_float2(12582912.0f, 12582912.0f);
  const float2 nmg = make_float2(-12582912.0f, -12582912.0f);
  const uint32_t w[4] = {v.x, v.y, v.z, v.w};
  float2 f[4], c[4];
  uint32_t tb[8];
  float dmax = 0.0f;
#pragma unroll
  for (int k = 0; k < 4; ++k) {
    f[k] = __half22float2(*reinterpret_cast<const __half2*>(&w[k]));
    const float2 q = __fmul2_rn(f[k], inv2);
    const float2 t = __fadd2_rn(q, mg);
    tb[2 * k] = __float_as_uint(t.x);
    tb[2 * k + 1] = __float_as_uint(t.y);
    c[k] = __fadd2_rn(t, nmg);
    const float2 d = __fadd2_rn(q, make_float2(-c[k].x, -c[k].y));
    dmax = fmaxf(dmax, fmaxf(fabsf(d.x), fabsf(d.y)));
  }
  if (dmax > 0.5f - 0x1p-17f) {
#pragma unroll
    for (int k = 0; k < 4; ++k) {
      c[k] = make_float2(rintf(__fdiv_rn(f[k].x, s)), rintf(__fdiv_rn(f[k].y, s)));
      tb[2 * k] = __float_as_uint(c[k].x + 12582912.0f);
      tb[2 * k + 1] = __float_as_uint(c[k].y + 12582912.0f);
    }
  }
#pragma unroll
  for (int k = 0; k < 4; ++k) n2 = __ffma2_rn(c[k], c[k], n2);
  // even-index codes in the low nibbles, odd-index codes in the high nibbles
  const uint32_t e = __byte_perm(__byte_perm(tb[0], tb[2], 0x0040), __byte_perm(tb[4], tb[6], 0x0040), 0x5410);
  const uint32_t o = __byte_perm(__byte_perm(tb[1], tb[3], 0x0040), __byte_perm(tb[5], tb[7], 0x0040), 0x5410);
  return (e & 0x0F0F0F0Fu) | ((o << 4) & 0xF0F0F0F0u);
}

// G warps quantize one row (8 / G rows per 256-thread CTA); each thread keeps
// up to MAXC 16-byte chunks of its row in registers between the abs-max and
// the quantization pass. Reductions are warp reductions, combined through
// shared memory when G > 1.
template <int G, int MAXC>
__global__ void __launch_bounds__(kThreads) quant_rows_kernel(RowSource src, int rows, int L, RowSinks out) {
  constexpr int kRowsPerCta = (kThreads / 32) / G;
  constexpr int kRowThreads = 32 * G;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int slot = warp / G;                           // row slot inside the CTA
  const int t = (warp % G) * 32 + lane;                // thread index inside the row
  const int row = blockIdx.x * kRowsPerCta + slot;
  const bool live = row < rows;
  const uint16_t* srow = nullptr;
  if (live) {
    if (src.idx == nullptr) {
      srow = src.X + static_cast<size_t>(row) * L;
    } else {
      const int per = src.K + src.T;
      const int b = row / per, r = row - b * per;
      if (r < src.K)
        srow = src.X + (static_cast<size_t>(b) * src.N + src.idx[b * src.K + r]) * L;
      else
        srow = src.text + (static_cast<size_t>(b) * src.T + (r - src.K)) * L;
    }
  }
  const int nch = L >> 3;
  const uint4* s4 = reinterpret_cast<const uint4*>(srow);

  uint4 v[MAXC];
  uint32_t m = 0;  // per-halfword max of |x| bit patterns (non-negative fp16 order as integers)
#pragma unroll
  for (int i = 0; i < MAXC; ++i) {
    const int c = t + i * kRowThreads;
    if (live && c < nch) {
      v[i] = __ldg(s4 + c);
      m = __vmaxu2(m, v[i].x & 0x7FFF7FFFu);
      m = __vmaxu2(m, v[i].y & 0x7FFF7FFFu);
      m = __vmaxu2(m, v[i].z & 0x7FFF7FFFu);
      m = __vmaxu2(m, v[i].w & 0x7FFF7FFFu);
    }
  }
  uint32_t mm = __reduce_max_sync(0xFFFFFFFFu, max(m & 0xFFFFu, m >> 16));
  __shared__ uint32_t red[kThreads / 32];
  __shared__ int red_n[kThreads / 32];
  if (G > 1) {
    if (lane == 0) red[warp] = mm;
    __syncthreads();
#pragma unroll
    for (int w = 0; w < G; ++w) mm = max(mm, red[slot * G + w]);
  }
  const float a = __half2float(__ushort_as_half(static_cast<unsigned short>(mm)));
  const float s = __fdiv_rn(a, 7.0f);
  const float inv = (a != 0.0f) ? __frcp_rn(s) : 0.0f;

  float2 n2 = make_float2(0.0f, 0.0f);  // exact: sums of squared codes <= 49 * 16384 < 2^24
  if (live) {
    uint32_t* q4 = reinterpret_cast<uint32_t*>(out.codes + static_cast<size_t>(row) * (L >> 1));
#pragma unroll
    for (int i = 0; i < MAXC; ++i) {
      const int c = t + i * kRowThreads;
      if (c < nch) {
        q4[c] = (a != 0.0f) ? quant_chunk(v[i], s, inv, n2) : 0u;
        if (out.copy) reinterpret_cast<uint4*>(out.copy + static_cast<size_t>(row) * L)[c] = v[i];
      }
    }
  }
  if (out.norm2) {
    int wn = __reduce_add_sync(0xFFFFFFFFu, static_cast<int>(n2.x + n2.y));
    if (G > 1) {
      if (lane == 0) red_n[warp] = wn;
      __syncthreads();
      wn = 0;
#pragma unroll
      for (int w = 0; w < G; ++w) wn += red_n[slot * G + w];
    }
    if (live && t == 0) out.norm2[row] = wn;
  }
  if (live && t == 0) out.scale[row] = (a != 0.0f) ? s : 0.0f;
}

template <int G, int MAXC>
cudaError_t launch_g(const RowSource& src, int rows, int L, const RowSinks& out, cudaStream_t stream) {
  constexpr int kRowsPerCta = (kThreads / 32) / G;
  quant_rows_kernel<G, MAXC><<<(rows + kRowsPerCta - 1) / kRowsPerCta, kThreads, 0, stream>>>(src, rows, L, out);
  return cudaGetLastError();
}

}  // namespace

cudaError_t launch_quant_rows(const RowSource& src, int rows, int L, const RowSinks& out,
                              cudaStream_t stream) {
  if (rows <= 0) return cudaSuccess;
  const int nch = L >> 3;  // 16-byte chunks per row
  if (nch <= 32 * 8) return launch_g<1, 8>(src, rows, L, out, stream);    // L <= 2048
  if (nch <= 32 * 20) return launch_g<1, 20>(src, rows, L, out, stream);  // L <= 5120
  if (nch <= 128 * 8) return launch_g<4, 8>(src, rows, L, out, stream);   // L <= 8192
  return launch_g<4, 16>(src, rows, L, out, stream);                      // L <= 16384
}

}  // namespace p4q
