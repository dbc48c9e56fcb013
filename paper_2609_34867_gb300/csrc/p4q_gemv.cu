// W4A4 linear for a few token rows (decode steps, small batches): the same
// exact integer products and dequantization as the GEMMs (App. A / App. B.3
// of the paper: per-token INT4 activations, per-output-channel INT4 weights,
// acc = sum_k a_k w_k exact, y = fp16_rne((float(acc) * s_a) * s_w)), for
// M <= 8 rows, where the weights are read once and the tensor cores would
// sit idle: the cost is streaming the packed weights from HBM.
//
// Kernel: the M activation rows are sign-extended once into shared memory,
// one byte per code (for each packed 32-bit word: its four low-nibble codes,
// then its four high-nibble codes; the weights use the same order, so every
// dot product is unchanged). Each warp streams whole weight rows, every lane
// a 16-byte chunk (32 codes) at a time, four chunks in flight (the next
// row's first ones while the current row is summed), sign-extends
// the chunk once and dp4a's it against every activation row; a warp sum per
// row gives the exact int32 accumulators, and lane m writes row m's output.
#include <cuda_fp16.h>

#include "p4q.h"
#include "p4q_device.cuh"
#include "p4q_internal.h"

namespace p4q {
namespace {

constexpr int kGemvWarps = 8;
constexpr int kGemvMaxRows = 8;  // above, the dp4a work per weight byte outweighs the stream
constexpr int kGemvUnroll = 4;                  // weight chunks in flight per lane
constexpr size_t kGemvSmemMax = 200u * 1024u;   // sign-extended activation rows

__device__ __forceinline__ int sext4(uint32_t n) {
  return static_cast<int>((n & 0x0F0F0F0Fu) | ((n & 0x08080808u) * 0x1Eu));
}

template <int MR, bool S32>
__global__ void __launch_bounds__(kGemvWarps * 32)
    gemv_w4a4_kernel(const uint8_t* __restrict__ Xq, const float* __restrict__ s_a, int M, int K,
                     const uint8_t* __restrict__ Wq, const float* __restrict__ s_w, int N, void* __restrict__ out) {
  pdl_wait();
  pdl_launch_dependents();
  extern __shared__ __align__(16) int8_t xs[];  // [M][K] sign-extended activation codes
  const int kb = K >> 1;                         // packed bytes per row
  const int nch = kb >> 4;                       // 16-byte packed chunks per row
  const int lane = threadIdx.x & 31;
  const int nwarps = gridDim.x * kGemvWarps;
  // the first weight chunks of this warp's first row are on their way while
  // the activations are staged
  int n = blockIdx.x * kGemvWarps + (threadIdx.x >> 5);
  uint4 wv[kGemvUnroll];
#pragma unroll
  for (int u = 0; u < kGemvUnroll; ++u) {
    const int c = lane + 32 * u;
    wv[u] = (n < N && c < nch) ? __ldg(reinterpret_cast<const uint4*>(Wq + static_cast<size_t>(n) * kb) + c)
                               : make_uint4(0u, 0u, 0u, 0u);
  }
  // stage the activations: 16 packed bytes -> 32 signed bytes
  for (int i = threadIdx.x; i < M * nch; i += blockDim.x) {
    const int m = i / nch, c = i - m * nch;
    const uint4 p = *reinterpret_cast<const uint4*>(Xq + static_cast<size_t>(m) * kb + 16 * c);
    const uint32_t w[4] = {p.x, p.y, p.z, p.w};
    int4* dst = reinterpret_cast<int4*>(xs + static_cast<size_t>(m) * K + 32 * c);
    dst[0] = make_int4(sext4(w[0]), sext4(w[0] >> 4), sext4(w[1]), sext4(w[1] >> 4));
    dst[1] = make_int4(sext4(w[2]), sext4(w[2] >> 4), sext4(w[3]), sext4(w[3] >> 4));
  }
  __syncthreads();
  for (; n < N; n += nwarps) {
    const uint4* wrow = reinterpret_cast<const uint4*>(Wq + static_cast<size_t>(n) * kb);
    int acc[MR];
#pragma unroll
    for (int m = 0; m < MR; ++m) acc[m] = 0;
    for (int c0 = lane; c0 < nch; c0 += 32 * kGemvUnroll) {
      if (c0 != lane) {  // the row's first chunks were loaded ahead
#pragma unroll
        for (int u = 0; u < kGemvUnroll; ++u) {
          const int c = c0 + 32 * u;
          wv[u] = c < nch ? __ldg(wrow + c) : make_uint4(0u, 0u, 0u, 0u);
        }
      }
#pragma unroll
      for (int u = 0; u < kGemvUnroll; ++u) {
        const int c = c0 + 32 * u;
        if (c >= nch) break;
        const uint32_t w[4] = {wv[u].x, wv[u].y, wv[u].z, wv[u].w};
        int e[8];
#pragma unroll
        for (int k = 0; k < 4; ++k) {
          e[2 * k] = sext4(w[k]);
          e[2 * k + 1] = sext4(w[k] >> 4);
        }
#pragma unroll
        for (int m = 0; m < MR; ++m) {
          if (m < M) {
            const int4* xr = reinterpret_cast<const int4*>(xs + static_cast<size_t>(m) * K + 32 * c);
            const int4 x0 = xr[0], x1 = xr[1];
            int a = acc[m];
            a = __dp4a(e[0], x0.x, a); a = __dp4a(e[1], x0.y, a); a = __dp4a(e[2], x0.z, a); a = __dp4a(e[3], x0.w, a);
            a = __dp4a(e[4], x1.x, a); a = __dp4a(e[5], x1.y, a); a = __dp4a(e[6], x1.z, a); a = __dp4a(e[7], x1.w, a);
            acc[m] = a;
          }
        }
      }
    }
    // the next row's first chunks go out before this row's sums
    const int nn = n + nwarps;
#pragma unroll
    for (int u = 0; u < kGemvUnroll; ++u) {
      const int c = lane + 32 * u;
      wv[u] = (nn < N && c < nch) ? __ldg(reinterpret_cast<const uint4*>(Wq + static_cast<size_t>(nn) * kb) + c)
                                  : make_uint4(0u, 0u, 0u, 0u);
    }
#pragma unroll
    for (int m = 0; m < MR; ++m) {
      if (m < M) {
        const int tot = __reduce_add_sync(0xFFFFFFFFu, acc[m]);
        if (lane == m) {
          if (S32) {
            static_cast<int32_t*>(out)[static_cast<size_t>(m) * N + n] = tot;
          } else {
            const float y = __fmul_rn(__fmul_rn(static_cast<float>(tot), s_a[m]), s_w[n]);
            static_cast<__half*>(out)[static_cast<size_t>(m) * N + n] = __float2half_rn(y);
          }
        }
      }
    }
  }
}

template <int MR, bool S32>
cudaError_t launch_mr(const GemmArgs& g, cudaStream_t stream) {
  const size_t smem = static_cast<size_t>(g.M) * g.K;
  static size_t smem_set = 48u << 10;
  if (smem > smem_set) {
    cudaError_t e = cudaFuncSetAttribute(gemv_w4a4_kernel<MR, S32>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         static_cast<int>(kGemvSmemMax));
    if (e != cudaSuccess) return e;
    smem_set = kGemvSmemMax;
  }
  // enough warps for every weight row, at most the CTAs that fit on the SMs
  const int per_sm = smem <= 24u * 1024u ? 8 : smem <= 48u * 1024u ? 4 : smem <= 100u * 1024u ? 2 : 1;
  const int want = (g.N + kGemvWarps - 1) / kGemvWarps;
  const int blocks = want < per_sm * num_sms() ? want : per_sm * num_sms();
  return launch_pdl(gemv_w4a4_kernel<MR, S32>, dim3(blocks), dim3(kGemvWarps * 32), smem, stream, g.A, g.s_a, g.M,
                    g.K, g.B, g.s_b, g.N, g.D);
}

template <bool S32>
cudaError_t launch_rows(const GemmArgs& g, cudaStream_t stream) {
  if (g.M <= 2) return launch_mr<2, S32>(g, stream);
  if (g.M <= 4) return launch_mr<4, S32>(g, stream);
  return launch_mr<8, S32>(g, stream);
}

}  // namespace

bool gemv_applies(const GemmArgs& g) {
  return (g.out == GemmOut::kHalf || g.out == GemmOut::kS32) && g.batch == 1 && g.M >= 1 && g.M <= kGemvMaxRows &&
         g.K % 32 == 0 && (g.d_pitch == 0 || g.d_pitch == g.N) && static_cast<size_t>(g.M) * g.K <= kGemvSmemMax;
}

cudaError_t launch_gemv(const GemmArgs& g, cudaStream_t stream) {
  return g.out == GemmOut::kS32 ? launch_rows<true>(g, stream) : launch_rows<false>(g, stream);
}

}  // namespace p4q
