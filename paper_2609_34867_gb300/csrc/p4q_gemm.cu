// W4A4 integer GEMM on the sm_103a tensor cores (tcgen05 + TMEM + TMA).
//
// Computes acc[m, n] = sum_k a[m, k] * b[n, k] exactly for INT4 codes a, b
// stored packed (two per byte, even index in the low nibble, two's
// complement), then applies one of three epilogues:
//   kHalf: y = fp16_rne(((float)acc * s_a[m]) * s_b[n])   (App. B.3 W4A4 linear)
//   kS32 : the int32 accumulators (test view)
//   kCos : (float)acc / sqrtf((float)na[m] * (float)nb[n])  (Eq. 4 CosSim of
//          two fake-quantized token rows, from their codes)
//
// The sm_103a tensor cores have no integer MMA kind, so the integer product is
// computed exactly on the FP8 path (tcgen05.mma kind::f8f6f4, E4M3 x E4M3 ->
// F32). Each 4-bit code v in [-8, 7] is stored in shared memory as the E4M3
// byte u = v + 8 in [0, 15]; the E4M3 bytes 0..15 encode exactly u * 2^-9
// (subnormals 0..7, then the first binade), so one nibble becomes one byte with
// a mask and an xor. The tensor core sums P = sum_k u_a u_b * 2^-18 in fp32;
// P * 2^18 < 225 * 16384 < 2^22 is an integer that fp32 holds exactly, and
//   acc = P - 8 * (sum_k u_a) - 8 * (sum_k u_b) + 64 K
// restores the signed product. The row sums of u are accumulated by the same
// threads that unpack the nibbles.
//
// Pipeline of one CTA (one 128 x BN output tile):
//   warp 0      TMA: packed tiles of A [128 x 64 B] and B [BN x 64 B] per
//               128-deep k-block into a ring of packed stages;
//   warps 2-9   unpack: packed stage -> E4M3 stage in the 128-byte swizzled
//               K-major layout the tensor core reads; also the row sums;
//   warp 1      MMA: 4 x tcgen05.mma (K = 32 each) per stage, accumulator in
//               TMEM (128 lanes x BN fp32 columns), commit frees the stage;
//   warps 2-5   epilogue: tcgen05.ld of the accumulator, correction, scaling,
//               store.
// The nibble order inside a 16-byte packed chunk is permuted identically for
// A and B (even k, then odd k), which leaves every dot product unchanged.
#include <cuda.h>
#include <cudaTypedefs.h>
#include <cuda_fp16.h>

#include <mutex>

#include "p4q_device.cuh"
#include "p4q_internal.h"

namespace p4q {
namespace {

__device__ unsigned int g_gemm_err;

constexpr int BM = 128;                      // tile rows (TMEM lanes)
constexpr int BK = 128;                      // k-elements per stage
constexpr int BKP = BK / 2;                  // packed bytes per row per stage
constexpr int kConvWarps = 8;
constexpr int kThreads = (2 + kConvWarps) * 32;
constexpr int kConvThreads = kConvWarps * 32;

template <int BN>
struct Cfg {
  static constexpr int SC = (BN == 256) ? 3 : 4;  // E4M3 stages
  static constexpr int SP = (BN == 256) ? 3 : 4;  // packed stages
  static constexpr int A_CONV = BM * BK;
  static constexpr int B_CONV = BN * BK;
  static constexpr int A_PACK = BM * BKP;
  static constexpr int B_PACK = BN * BKP;
  static constexpr int CONV_STAGE = A_CONV + B_CONV;
  static constexpr int PACK_STAGE = A_PACK + B_PACK;
  static constexpr int OFF_PACK = SC * CONV_STAGE;
  static constexpr int OFF_BAR = OFF_PACK + SP * PACK_STAGE;
  static constexpr int NBAR = 2 * SP + 2 * SC + 2;
  static constexpr int OFF_MISC = OFF_BAR + NBAR * 8;      // tmem slot, abort flag
  static constexpr int OFF_SUM = OFF_MISC + 16;
  static constexpr int SMEM = 1024 + OFF_SUM + (BM + BN) * 4;
  static constexpr uint32_t TMEM_COLS = BN;
};

struct Params {
  int M, N, K;
  int out;  // GemmOut
  void* D;
  const float* s_a;
  const float* s_b;
  const int32_t* norm_a;
  const int32_t* norm_b;
};

__device__ __forceinline__ uint32_t nib_lo(uint32_t w) { return (w & 0x0F0F0F0Fu) ^ 0x08080808u; }
__device__ __forceinline__ uint32_t nib_hi(uint32_t w) { return ((w >> 4) & 0x0F0F0F0Fu) ^ 0x08080808u; }

// Unpacks one 16-byte packed chunk (32 codes of one row) into 32 E4M3 bytes at
// logical byte offset 32*c of row r of a 128-byte-swizzled K-major tile, and
// returns the sum of the 32 offset codes u.
__device__ __forceinline__ int unpack_chunk(const uint8_t* pack_row, uint8_t* conv_tile, int r, int c) {
  const uint4 p = *reinterpret_cast<const uint4*>(pack_row + c * 16);
  const uint32_t l0 = nib_lo(p.x), h0 = nib_hi(p.x), l1 = nib_lo(p.y), h1 = nib_hi(p.y);
  const uint32_t l2 = nib_lo(p.z), h2 = nib_hi(p.z), l3 = nib_lo(p.w), h3 = nib_hi(p.w);
  uint8_t* row = conv_tile + r * 128;
  const int sw = r & 7;
  *reinterpret_cast<uint4*>(row + (((2 * c) ^ sw) << 4)) = make_uint4(l0, h0, l1, h1);
  *reinterpret_cast<uint4*>(row + (((2 * c + 1) ^ sw) << 4)) = make_uint4(l2, h2, l3, h3);
  const uint32_t bytesum = l0 + h0 + l1 + h1 + l2 + h2 + l3 + h3;  // <= 8 * 15 per byte
  return __dp4a(bytesum, 0x01010101u, 0u);
}

template <int BN>
__global__ void __launch_bounds__(kThreads, 1)
    w4a4_gemm_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB,
                     const Params p) {
  using C = Cfg<BN>;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + C::OFF_BAR);
  uint64_t* full_p = bars;
  uint64_t* empty_p = bars + C::SP;
  uint64_t* full_c = bars + 2 * C::SP;
  uint64_t* empty_c = bars + 2 * C::SP + C::SC;
  uint64_t* acc_full = bars + 2 * C::SP + 2 * C::SC;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(smem + C::OFF_MISC);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(smem + C::OFF_MISC + 4);
  int* sumA = reinterpret_cast<int*>(smem + C::OFF_SUM);
  int* sumB = sumA + BM;

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int n0 = blockIdx.x * BN, m0 = blockIdx.y * BM, bz = blockIdx.z;
  const int KB = p.K / BK;

  if (threadIdx.x == 0) {
    for (int i = 0; i < C::SP; ++i) {
      mbar_init(&full_p[i], 1);
      mbar_init(&empty_p[i], kConvWarps);
    }
    for (int i = 0; i < C::SC; ++i) {
      mbar_init(&full_c[i], kConvWarps);
      mbar_init(&empty_c[i], 1);
    }
    mbar_init(acc_full, 1);
    *abort_flag = 0;
    fence_barrier_init();
  }
  if (warp == 1) {
    tmem_alloc(tmem_slot, C::TMEM_COLS);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem_base = *tmem_slot;

  if (warp == 0) {
    if (lane == 0) {
      tma_prefetch_desc(&tmA);
      tma_prefetch_desc(&tmB);
      int issued = 0;
      for (int kb = 0; kb < KB; ++kb) {
        const int s = kb % C::SP;
        const uint32_t ph = (kb / C::SP) & 1;
        if (!mbar_wait(&empty_p[s], ph ^ 1, abort_flag, &g_gemm_err)) break;
        uint8_t* pa = smem + C::OFF_PACK + s * C::PACK_STAGE;
        mbar_arrive_expect_tx(&full_p[s], C::PACK_STAGE);
        tma_load_3d(&tmA, &full_p[s], pa, kb * BKP, m0, bz);
        tma_load_3d(&tmB, &full_p[s], pa + C::A_PACK, kb * BKP, n0, bz);
        issued = kb + 1;
      }
      if (*abort_flag) {
        // Let the copies already in flight land before the CTA exits.
        for (int kb = max(0, issued - C::SP); kb < issued; ++kb) {
          const uint32_t a = smem_u32(&full_p[kb % C::SP]);
          const unsigned long long t0 = globaltimer();
          while (!mbar_try_wait(a, (kb / C::SP) & 1) && globaltimer() - t0 < 100000000ull) {
          }
        }
      }
    }
  } else if (warp == 1) {
    if (lane == 0) {
      constexpr uint32_t idesc = idesc_e4m3_f32(BM, BN);
      for (int kb = 0; kb < KB; ++kb) {
        const int t = kb % C::SC;
        const uint32_t ph = (kb / C::SC) & 1;
        if (!mbar_wait(&full_c[t], ph, abort_flag, &g_gemm_err)) break;
        tc_fence_after();
        const uint32_t a0 = smem_u32(smem + t * C::CONV_STAGE);
        const uint32_t b0 = a0 + C::A_CONV;
#pragma unroll
        for (int k = 0; k < BK / 32; ++k)
          mma_f8f6f4(tmem_base, sw128_kmajor_desc(a0 + k * 32), sw128_kmajor_desc(b0 + k * 32), idesc,
                     (kb | k) != 0 ? 1u : 0u);
        mma_commit(&empty_c[t]);
      }
      mma_commit(acc_full);
    }
  } else {
    // ---------------- unpack warps
    const int tc = threadIdx.x - 64;
    int accA[BM * 4 / kConvThreads];
    int accB[BN * 4 / kConvThreads];
#pragma unroll
    for (int j = 0; j < BM * 4 / kConvThreads; ++j) accA[j] = 0;
#pragma unroll
    for (int j = 0; j < BN * 4 / kConvThreads; ++j) accB[j] = 0;
    for (int kb = 0; kb < KB; ++kb) {
      const int s = kb % C::SP, t = kb % C::SC;
      if (!mbar_wait(&full_p[s], (kb / C::SP) & 1, abort_flag, &g_gemm_err)) break;
      if (!mbar_wait(&empty_c[t], ((kb / C::SC) & 1) ^ 1, abort_flag, &g_gemm_err)) break;
      const uint8_t* pa = smem + C::OFF_PACK + s * C::PACK_STAGE;
      const uint8_t* pb = pa + C::A_PACK;
      uint8_t* ca = smem + t * C::CONV_STAGE;
      uint8_t* cb = ca + C::A_CONV;
#pragma unroll
      for (int j = 0; j < BM * 4 / kConvThreads; ++j) {
        const int task = tc + j * kConvThreads;
        const int r = task >> 2, c = task & 3;
        accA[j] += unpack_chunk(pa + r * BKP, ca, r, c);
      }
#pragma unroll
      for (int j = 0; j < BN * 4 / kConvThreads; ++j) {
        const int task = tc + j * kConvThreads;
        const int r = task >> 2, c = task & 3;
        accB[j] += unpack_chunk(pb + r * BKP, cb, r, c);
      }
      fence_proxy_async_smem();
      __syncwarp();
      if (lane == 0) {
        mbar_arrive(&empty_p[s]);
        mbar_arrive(&full_c[t]);
      }
    }
    // row sums of u over the whole K: reduce the 4 threads sharing a row
#pragma unroll
    for (int j = 0; j < BM * 4 / kConvThreads; ++j) {
      int v = accA[j];
      v += __shfl_xor_sync(0xFFFFFFFFu, v, 1);
      v += __shfl_xor_sync(0xFFFFFFFFu, v, 2);
      if ((tc & 3) == 0) sumA[(tc + j * kConvThreads) >> 2] = v;
    }
#pragma unroll
    for (int j = 0; j < BN * 4 / kConvThreads; ++j) {
      int v = accB[j];
      v += __shfl_xor_sync(0xFFFFFFFFu, v, 1);
      v += __shfl_xor_sync(0xFFFFFFFFu, v, 2);
      if ((tc & 3) == 0) sumB[(tc + j * kConvThreads) >> 2] = v;
    }
    asm volatile("bar.sync 1, %0;" ::"r"(kConvThreads) : "memory");

    if (warp < 6) {
      // ---------------- epilogue: warps 2..5 cover TMEM lane quarters 2,3,0,1
      const bool ok = mbar_wait(acc_full, 0, abort_flag, &g_gemm_err);
      tc_fence_after();
      const int q = warp & 3;
      const int row = q * 32 + lane;
      const int m = m0 + row;
      const int corrA = 64 * p.K - 8 * sumA[row];
      float sa = 0.0f;
      int na = 0;
      if (ok && m < p.M) {
        if (p.out == static_cast<int>(GemmOut::kHalf)) sa = p.s_a[m];
        if (p.out == static_cast<int>(GemmOut::kCos)) na = p.norm_a[static_cast<size_t>(bz) * p.M + m];
      }
#pragma unroll 1
      for (int cc = 0; cc < BN / 32; ++cc) {
        uint32_t r[32];
        tmem_ld_32x32b_x32(tmem_base + (static_cast<uint32_t>(q * 32) << 16) + cc * 32, r);
        tmem_ld_wait();
        const int nb = n0 + cc * 32;
        if (!ok || m >= p.M || nb >= p.N) continue;
        int acc[32];
#pragma unroll
        for (int i = 0; i < 32; ++i) {
          const int P = __float2int_rn(__uint_as_float(r[i]) * 262144.0f);
          acc[i] = P + corrA - 8 * sumB[cc * 32 + i];
        }
        const size_t base = (static_cast<size_t>(bz) * p.M + m) * p.N + nb;
        if (p.out == static_cast<int>(GemmOut::kHalf)) {
          __half* y = reinterpret_cast<__half*>(p.D) + base;
#pragma unroll
          for (int g = 0; g < 4; ++g) {
            if (nb + g * 8 >= p.N) break;
            uint32_t w[4];
#pragma unroll
            for (int e = 0; e < 4; ++e) {
              const int i0 = g * 8 + 2 * e;
              const float y0 = __fmul_rn(__fmul_rn(static_cast<float>(acc[i0]), sa), p.s_b[nb + i0]);
              const float y1 = __fmul_rn(__fmul_rn(static_cast<float>(acc[i0 + 1]), sa), p.s_b[nb + i0 + 1]);
              const __half2 h = __floats2half2_rn(y0, y1);
              w[e] = *reinterpret_cast<const uint32_t*>(&h);
            }
            *reinterpret_cast<uint4*>(y + g * 8) = make_uint4(w[0], w[1], w[2], w[3]);
          }
        } else if (p.out == static_cast<int>(GemmOut::kS32)) {
          int32_t* y = reinterpret_cast<int32_t*>(p.D) + base;
#pragma unroll
          for (int g = 0; g < 8; ++g) {
            if (nb + g * 4 >= p.N) break;
            *reinterpret_cast<int4*>(y + g * 4) = make_int4(acc[g * 4], acc[g * 4 + 1], acc[g * 4 + 2], acc[g * 4 + 3]);
          }
        } else {
          // Token counts need not be multiples of 4: vector stores only when
          // every row of the output starts on a 16-byte boundary.
          float* y = reinterpret_cast<float*>(p.D) + base;
          const int32_t* nbv = p.norm_b + static_cast<size_t>(bz) * p.N;
          const int ncol = min(32, p.N - nb);
          float o[32];
#pragma unroll
          for (int i = 0; i < 32; ++i) {
            const int nn = (i < ncol) ? nbv[nb + i] : 0;
            o[i] = (na == 0 || nn == 0)
                       ? 0.0f
                       : __fdiv_rn(static_cast<float>(acc[i]),
                                   __fsqrt_rn(__fmul_rn(static_cast<float>(na), static_cast<float>(nn))));
          }
          if ((p.N & 3) == 0) {
#pragma unroll
            for (int g = 0; g < 8; ++g)
              if (g * 4 < ncol) *reinterpret_cast<float4*>(y + g * 4) = make_float4(o[g * 4], o[g * 4 + 1], o[g * 4 + 2], o[g * 4 + 3]);
          } else {
#pragma unroll
            for (int i = 0; i < 32; ++i)
              if (i < ncol) y[i] = o[i];
          }
        }
      }
    }
  }

  // Teardown: every MMA must have completed before TMEM is released.
  if (warp == 1 && lane == 0 && *abort_flag) {
    const uint32_t a = smem_u32(acc_full);
    const unsigned long long t0 = globaltimer();
    while (!mbar_try_wait(a, 0) && globaltimer() - t0 < 100000000ull) {
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem_base, C::TMEM_COLS);
  }
}

PFN_cuTensorMapEncodeTiled_v12000 get_encode_fn() {
  static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void* ptr = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &ptr, 12000, cudaEnableDefault, &q) ==
            cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(ptr);
  });
  return fn;
}

// 3-D map over packed rows: dims (K/2 bytes, rows, batch), box (64, box_rows, 1).
bool make_map(CUtensorMap* map, const uint8_t* base, int K, int rows, int batch, long long batch_stride_rows,
              int box_rows) {
  auto enc = get_encode_fn();
  if (!enc) return false;
  const cuuint64_t kb = static_cast<cuuint64_t>(K / 2);
  cuuint64_t dims[3] = {kb, static_cast<cuuint64_t>(rows), static_cast<cuuint64_t>(batch)};
  const long long bs = batch_stride_rows > 0 ? batch_stride_rows : rows;
  cuuint64_t strides[2] = {kb, static_cast<cuuint64_t>(bs) * kb};
  cuuint32_t box[3] = {static_cast<cuuint32_t>(BKP), static_cast<cuuint32_t>(box_rows), 1};
  cuuint32_t estr[3] = {1, 1, 1};
  CUresult r = enc(map, CU_TENSOR_MAP_DATA_TYPE_UINT8, 3, const_cast<uint8_t*>(base), dims, strides, box, estr,
                   CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_NONE, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                   CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS;
}

template <int BN>
cudaError_t launch_bn(const GemmArgs& g, cudaStream_t stream) {
  using C = Cfg<BN>;
  static bool attr_set = false;
  if (!attr_set) {
    cudaError_t e = cudaFuncSetAttribute(w4a4_gemm_kernel<BN>, cudaFuncAttributeMaxDynamicSharedMemorySize, C::SMEM);
    if (e != cudaSuccess) return e;
    attr_set = true;
  }
  CUtensorMap ma, mb;
  if (!make_map(&ma, g.A, g.K, g.M, g.batch, g.a_batch_stride, BM)) return cudaErrorInvalidValue;
  if (!make_map(&mb, g.B, g.K, g.N, g.batch, g.b_batch_stride, BN)) return cudaErrorInvalidValue;
  Params p{g.M, g.N, g.K, static_cast<int>(g.out), g.D, g.s_a, g.s_b, g.norm_a, g.norm_b};
  dim3 grid((g.N + BN - 1) / BN, (g.M + BM - 1) / BM, g.batch);
  w4a4_gemm_kernel<BN><<<grid, kThreads, C::SMEM, stream>>>(ma, mb, p);
  return cudaGetLastError();
}

}  // namespace

cudaError_t launch_w4a4_gemm(const GemmArgs& g, cudaStream_t stream) {
  if (g.M <= 0 || g.N <= 0 || g.batch <= 0) return cudaSuccess;
  if (g.N >= 1024 && g.out != GemmOut::kCos) return launch_bn<256>(g, stream);
  return launch_bn<128>(g, stream);
}

unsigned int gemm_read_and_clear_error() {
  unsigned int v = 0, z = 0;
  cudaMemcpyFromSymbol(&v, g_gemm_err, sizeof(v));
  cudaMemcpyToSymbol(g_gemm_err, &z, sizeof(z));
  return v;
}

}  // namespace p4q
