// Throughput probes that give the roofline denominators of the integer
// contractions (the paper has no counterpart; nothing of the hot path runs
// here). Each kernel keeps one pipe busy with independent work whose operands
// stay on chip, so its time measures the pipe's sustainable rate on this GPU:
//   kind 0  tcgen05.mma.cta_group::2.kind::f8f6f4 (E4M3 x E4M3 -> F32,
//           M 256 x N 256 x K 32 per instruction), operands in shared memory,
//           one CTA pair per two SMs: the pipe the exact INT4 GEMM runs on;
//   kind 1  mma.sync.aligned.m16n8k32 s8 x s8 -> s32 (the legacy warp-level
//           integer tensor path), eight independent accumulators per warp;
//   kind 2  dp4a (four s8 products summed into an s32, CUDA cores), eight
//           independent chains per thread.
// Operand values are codes of the same range the GEMM multiplies (bytes 0..15
// for the FP8 probe, -8..7 for the integer probes), drawn per thread from a
// hash, since the energy per operation and thus the clock under load depend
// on the data.
#include <cuda_runtime.h>

#include "p4q_device.cuh"
#include "p4q_internal.h"

namespace p4q {

__device__ unsigned int g_peak_err;

namespace {

constexpr int kTcThreads = 128;
constexpr int kTcTileBytes = 128 * 128;  // 128 rows x 128 bytes (K = 128) per operand and CTA
constexpr uint32_t kTcCols = 256;

__device__ __forceinline__ uint32_t mix32(uint32_t x) {
  x ^= x >> 16;
  x *= 0x7FEB352Du;
  x ^= x >> 15;
  x *= 0x846CA68Bu;
  x ^= x >> 16;
  return x;
}

// One cluster of two CTAs: each holds 128 rows of A and 128 rows of B for one
// 128-deep k-block in the 128-byte-swizzled K-major layout (any byte order is
// a valid operand), and the leader issues `iters` x 4 MMAs of M 256 x N 256 x
// K 32 into one TMEM accumulator, then one commit.
__global__ void __cluster_dims__(2, 1, 1) __launch_bounds__(kTcThreads, 1)
    tc_peak_kernel(int iters, uint32_t* __restrict__ sink) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint8_t* a = smem;
  uint8_t* b = smem + kTcTileBytes;
  uint64_t* done = reinterpret_cast<uint64_t*>(smem + 2 * kTcTileBytes);
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(smem + 2 * kTcTileBytes + 8);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(smem + 2 * kTcTileBytes + 12);
  const int warp = threadIdx.x >> 5;
  const uint32_t rank = cluster_ctarank();
  const uint32_t seed = (blockIdx.x + 1u) * 0x9E3779B9u;
  for (int i = threadIdx.x; i < 2 * kTcTileBytes / 4; i += kTcThreads) {
    const uint32_t h = mix32(seed ^ static_cast<uint32_t>(i));
    reinterpret_cast<uint32_t*>(smem)[i] = h & 0x0F0F0F0Fu;  // four bytes in 0..15
  }
  if (threadIdx.x == 0) {
    mbar_init(done, 1);
    *abort_flag = 0;
    fence_barrier_init();
  }
  fence_proxy_async_smem();  // the operand bytes were written by the generic proxy
  if (warp == 0) {
    tmem_alloc_pair(tmem_slot, kTcCols);
    tmem_relinquish_pair();
  }
  tc_fence_before();
  cluster_sync();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  pdl_wait();
  if (threadIdx.x == 0 && rank == 0) {
    constexpr uint32_t idesc = idesc_e4m3_f32(256, 256);
    const uint32_t a0 = smem_u32(a), b0 = smem_u32(b);
    for (int it = 0; it < iters; ++it) {
#pragma unroll
      for (int k = 0; k < 4; ++k)
        mma_f8f6f4_pair(tmem, sw128_kmajor_desc(a0 + 32 * k), sw128_kmajor_desc(b0 + 32 * k), idesc,
                        (it | k) != 0 ? 1u : 0u);
    }
    mma_commit_pair(done, 3);
  }
  // both CTAs' barriers receive the multicast commit
  if (threadIdx.x == 0) {
    if (!mbar_wait(done, 0, abort_flag, &g_peak_err)) *abort_flag = 1;
  }
  __syncthreads();
  tc_fence_after();
  if (warp == 0) {
    uint32_t v[16];
    tmem_ld_32x32b_x16(tmem, v);
    tmem_ld_wait();
    uint32_t x = 0;
#pragma unroll
    for (int i = 0; i < 16; ++i) x ^= v[i];
    if (x == 0x7FC00001u) sink[blockIdx.x] = x;  // never true in practice; keeps the result live
  }
  tc_fence_before();
  cluster_sync();
  if (warp == 0) {
    tc_fence_after();
    tmem_dealloc_pair(tmem, kTcCols);
  }
}

constexpr int kChains = 8;

// The low nibble of each byte of x as a two's complement 4-bit code, sign-extended to the byte (-8..7).
__device__ __forceinline__ uint32_t sext4(uint32_t x) { return (x & 0x0F0F0F0Fu) | ((x & 0x08080808u) * 0x1Eu); }

// kind 1: m16n8k32 s8 MMAs on register operands, kChains independent accumulators per warp.
__global__ void __launch_bounds__(256) s8_mma_peak_kernel(int iters, uint32_t* __restrict__ sink) {
  pdl_wait();
  const uint32_t h = mix32(blockIdx.x * 256u + threadIdx.x);
  const uint32_t a0 = sext4(h), a1 = sext4(h >> 4);
  const uint32_t b0 = sext4(mix32(h)), b1 = sext4(mix32(h) >> 4);
  int c[kChains][4];
#pragma unroll
  for (int j = 0; j < kChains; ++j) c[j][0] = c[j][1] = c[j][2] = c[j][3] = j;
  for (int it = 0; it < iters; ++it) {
#pragma unroll
    for (int j = 0; j < kChains; ++j) {
      asm volatile(
          "mma.sync.aligned.m16n8k32.row.col.s32.s8.s8.s32 {%0, %1, %2, %3}, {%4, %5, %6, %7}, {%8, %9}, "
          "{%0, %1, %2, %3};"
          : "+r"(c[j][0]), "+r"(c[j][1]), "+r"(c[j][2]), "+r"(c[j][3])
          : "r"(a0), "r"(a1), "r"(a1), "r"(a0), "r"(b0), "r"(b1));
    }
  }
  int x = 0;
#pragma unroll
  for (int j = 0; j < kChains; ++j) x ^= c[j][0] ^ c[j][1] ^ c[j][2] ^ c[j][3];
  if (x == 0x5EED1234) sink[blockIdx.x] = static_cast<uint32_t>(x);
}

// kind 2: dp4a, kChains independent chains per thread.
__global__ void __launch_bounds__(256) dp4a_peak_kernel(int iters, uint32_t* __restrict__ sink) {
  pdl_wait();
  const uint32_t h = mix32(blockIdx.x * 256u + threadIdx.x);
  const int a = static_cast<int>(sext4(h)), b = static_cast<int>(sext4(mix32(h)));
  int c[kChains];
#pragma unroll
  for (int j = 0; j < kChains; ++j) c[j] = j;
  for (int it = 0; it < iters; ++it) {
#pragma unroll
    for (int j = 0; j < kChains; ++j) c[j] = __dp4a(a, b ^ (j << 8), c[j]);
  }
  int x = 0;
#pragma unroll
  for (int j = 0; j < kChains; ++j) x ^= c[j];
  if (x == 0x5EED1234) sink[blockIdx.x] = static_cast<uint32_t>(x);
}

}  // namespace

size_t peak_probe_sink_words() { return 8 * 1024; }

cudaError_t launch_peak_probe(int kind, int iters, uint32_t* sink, double* ops, cudaStream_t stream) {
  const int sms = num_sms();
  if (kind == 0) {
    static bool attr_set = false;
    const int smem = 1024 + 2 * kTcTileBytes + 64;
    if (!attr_set) {
      cudaError_t e = cudaFuncSetAttribute(tc_peak_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
      if (e != cudaSuccess) return e;
      attr_set = true;
    }
    const int ctas = 2 * (sms / 2);
    *ops = 2.0 * 256 * 256 * 32 * 4.0 * iters * (ctas / 2);
    return launch_pdl(tc_peak_kernel, dim3(ctas), dim3(kTcThreads), smem, stream, iters, sink);
  }
  const int blocks = 4 * sms;  // 32 warps per SM
  if (kind == 1) {
    *ops = 2.0 * 16 * 8 * 32 * kChains * static_cast<double>(iters) * blocks * 8;
    return launch_pdl(s8_mma_peak_kernel, dim3(blocks), dim3(256), 0, stream, iters, sink);
  }
  *ops = 8.0 * kChains * static_cast<double>(iters) * blocks * 256;
  return launch_pdl(dp4a_peak_kernel, dim3(blocks), dim3(256), 0, stream, iters, sink);
}

unsigned int peak_read_and_clear_error() {
  unsigned int v = 0, z = 0;
  cudaMemcpyFromSymbol(&v, g_peak_err, sizeof(v));
  cudaMemcpyToSymbol(g_peak_err, &z, sizeof(z));
  return v;
}

}  // namespace p4q
