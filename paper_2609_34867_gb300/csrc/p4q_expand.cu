// Expansion of packed INT4 codes to one byte per code (u = v + 8, the E4M3
// byte the FP8 MMAs read exactly as u * 2^-9) with the per-row sums of u:
// the operands of the expanded-operand GEMM (p4q_gemm8.cu). HBM-bound
// streaming kernel: bytes per row K/2 in, K + 4 out.
#include "p4q_device.cuh"
#include "p4q_internal.h"

namespace p4q {
namespace {

// One warp per row: packed codes [rows, K/2] -> one byte per code u = v + 8
// [rows, K] (per packed 32-bit word: its four low-nibble codes, then its four
// high-nibble codes) and sum_u[row]. All of a lane's 16-byte loads of the row
// are issued before the first store (MAXC chunks per lane).
template <int MAXC>
__global__ void __launch_bounds__(256) expand_codes_kernel(const uint8_t* __restrict__ src, int rows, int K,
                                                           uint8_t* __restrict__ dst, int32_t* __restrict__ sums) {
  pdl_wait();
  pdl_launch_dependents();
  const int row = blockIdx.x * 8 + (threadIdx.x >> 5), lane = threadIdx.x & 31;
  if (row >= rows) return;
  const uint4* s4 = reinterpret_cast<const uint4*>(src + static_cast<size_t>(row) * (K >> 1));
  uint4* d4 = reinterpret_cast<uint4*>(dst + static_cast<size_t>(row) * K);
  const int nch = K >> 5;  // 16-byte packed chunks per row
  uint4 w[MAXC];
#pragma unroll
  for (int i = 0; i < MAXC; ++i) {
    const int c = lane + 32 * i;
    if (c < nch) w[i] = ldg_stream16(s4 + c);
  }
  constexpr uint32_t ones = 0x01010101u;
  uint32_t acc = 0;
#pragma unroll
  for (int i = 0; i < MAXC; ++i) {
    const int c = lane + 32 * i;
    if (c < nch) {
      const uint32_t l0 = (w[i].x & 0x0F0F0F0Fu) ^ 0x08080808u, h0 = ((w[i].x >> 4) & 0x0F0F0F0Fu) ^ 0x08080808u;
      const uint32_t l1 = (w[i].y & 0x0F0F0F0Fu) ^ 0x08080808u, h1 = ((w[i].y >> 4) & 0x0F0F0F0Fu) ^ 0x08080808u;
      const uint32_t l2 = (w[i].z & 0x0F0F0F0Fu) ^ 0x08080808u, h2 = ((w[i].z >> 4) & 0x0F0F0F0Fu) ^ 0x08080808u;
      const uint32_t l3 = (w[i].w & 0x0F0F0F0Fu) ^ 0x08080808u, h3 = ((w[i].w >> 4) & 0x0F0F0F0Fu) ^ 0x08080808u;
      d4[2 * c] = make_uint4(l0, h0, l1, h1);
      d4[2 * c + 1] = make_uint4(l2, h2, l3, h3);
      // byte-wise sum of the eight words first (each byte <= 8 x 15 < 256), then one dp4a
      acc = __dp4a(l0 + h0 + l1 + h1 + l2 + h2 + l3 + h3, ones, acc);
    }
  }
  acc = __reduce_add_sync(0xFFFFFFFFu, acc);
  if (lane == 0) sums[row] = static_cast<int32_t>(acc);
}

}  // namespace

cudaError_t launch_expand_codes(const uint8_t* q, int rows, int K, uint8_t* u, int32_t* sum_u, cudaStream_t stream) {
  if (rows <= 0) return cudaSuccess;
  const dim3 grid((rows + 7) / 8), block(256);
  const int nch = K >> 5;
  if (nch <= 32 * 4) return launch_pdl(expand_codes_kernel<4>, grid, block, 0, stream, q, rows, K, u, sum_u);
  if (nch <= 32 * 8) return launch_pdl(expand_codes_kernel<8>, grid, block, 0, stream, q, rows, K, u, sum_u);
  return launch_pdl(expand_codes_kernel<16>, grid, block, 0, stream, q, rows, K, u, sum_u);
}

}  // namespace p4q
