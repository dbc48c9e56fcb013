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
// P * 2^18 <= 225 * 16384 < 2^22 is an integer that fp32 holds exactly, and
//   acc = P - 8 * (sum_k u_a) - 8 * (sum_k u_b) + 64 K
// restores the signed product. The row sums of u are accumulated by the same
// threads that unpack the nibbles.
//
// Persistent kernel, one CTA per SM, static round-robin over output tiles
// (m fastest, so CTAs running together share the same B tile in L2):
//   warp 0       TMA: packed tiles of A [128 x 64 B] and B [BN x 64 B] per
//                128-deep k-block into a ring of SP packed stages;
//   warps 2-9    unpack: packed stage -> E4M3 stage in the 128-byte swizzled
//                K-major layout the tensor core reads (ring of SC stages),
//                plus the per-row sums of u for the correction;
//   warp 1       MMA: 4 x tcgen05.mma (K = 32 each) per k-block into one of
//                two TMEM accumulators (128 lanes x BN fp32 columns each);
//   warps 10-13  epilogue of the previous tile, overlapped with the next
//                tile's main loop: tcgen05.ld, correction, scaling, a 32 x 32
//                box staged in swizzled shared memory, TMA store.
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
constexpr int kEpiWarps = 4;
constexpr int kConvThreads = kConvWarps * 32;
constexpr int kFirstConvWarp = 2;
constexpr int kFirstEpiWarp = kFirstConvWarp + kConvWarps;
constexpr int kThreads = (kFirstEpiWarp + kEpiWarps) * 32;

template <int BN, int MODE>
struct Cfg {
  static constexpr int SC = (BN == 256) ? 2 : 3;  // E4M3 stages
  static constexpr int SP = (BN == 256) ? 4 : 5;  // packed stages
  static constexpr int A_CONV = BM * BK;
  static constexpr int B_CONV = BN * BK;
  static constexpr int A_PACK = BM * BKP;
  static constexpr int B_PACK = BN * BKP;
  static constexpr int CONV_STAGE = A_CONV + B_CONV;
  static constexpr int PACK_STAGE = A_PACK + B_PACK;
  static constexpr int ELEM = (MODE == static_cast<int>(GemmOut::kHalf)) ? 2 : 4;
  static constexpr int BOX_BYTES = 32 * 32 * ELEM;  // one 32 x 32 output box
  static constexpr int OFF_PACK = SC * CONV_STAGE;
  static constexpr int OFF_STAGE = OFF_PACK + SP * PACK_STAGE;  // epilogue boxes, 2 per warp
  static constexpr int OFF_SUMA = OFF_STAGE + kEpiWarps * 2 * BOX_BYTES;
  static constexpr int OFF_SUMB = OFF_SUMA + 2 * BM * 4;
  static constexpr int OFF_SCOL = OFF_SUMB + 2 * BN * 4;           // per-warp column scale / norm cache
  static constexpr int OFF_BAR = OFF_SCOL + kEpiWarps * BN * 4;
  static constexpr int NBAR = 2 * SP + 2 * SC + 8;
  static constexpr int OFF_MISC = OFF_BAR + NBAR * 8;
  static constexpr int SMEM = 1024 + OFF_MISC + 16;
  static constexpr uint32_t TMEM_COLS = 2 * BN;
  static_assert(SMEM <= 232448, "shared memory budget");
};

struct Params {
  int M, N, K, batch;
  int num_m, num_n, tiles;
  const float* s_a;
  const float* s_b;
  const int32_t* norm_a;
  const int32_t* norm_b;
};

__device__ __forceinline__ uint32_t nib_lo(uint32_t w) { return (w & 0x0F0F0F0Fu) ^ 0x08080808u; }
__device__ __forceinline__ uint32_t nib_hi(uint32_t w) { return ((w >> 4) & 0x0F0F0F0Fu) ^ 0x08080808u; }

// Writes the 32 E4M3 bytes of one 16-byte packed chunk (32 codes of one row)
// at logical byte offset 32*c of row r of a 128-byte-swizzled K-major tile and
// returns the sum of the 32 offset codes u.
__device__ __forceinline__ int convert_chunk(const uint4 p, uint8_t* conv_tile, int r, int c) {
  const uint32_t l0 = nib_lo(p.x), h0 = nib_hi(p.x), l1 = nib_lo(p.y), h1 = nib_hi(p.y);
  const uint32_t l2 = nib_lo(p.z), h2 = nib_hi(p.z), l3 = nib_lo(p.w), h3 = nib_hi(p.w);
  uint8_t* row = conv_tile + r * 128;
  const int sw = r & 7;
  *reinterpret_cast<uint4*>(row + (((2 * c) ^ sw) << 4)) = make_uint4(l0, h0, l1, h1);
  *reinterpret_cast<uint4*>(row + (((2 * c + 1) ^ sw) << 4)) = make_uint4(l2, h2, l3, h3);
  const uint32_t bytesum = l0 + h0 + l1 + h1 + l2 + h2 + l3 + h3;  // <= 8 * 15 per byte
  return __dp4a(bytesum, 0x01010101u, 0u);
}

template <int BN, int MODE>
__global__ void __launch_bounds__(kThreads, 1)
    w4a4_gemm_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB,
                     const __grid_constant__ CUtensorMap tmD, const Params p) {
  using C = Cfg<BN, MODE>;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + C::OFF_BAR);
  uint64_t* full_p = bars;                        // TMA -> unpack
  uint64_t* empty_p = full_p + C::SP;             // unpack -> TMA
  uint64_t* full_c = empty_p + C::SP;             // unpack -> MMA
  uint64_t* empty_c = full_c + C::SC;             // MMA -> unpack
  uint64_t* acc_full = empty_c + C::SC;           // [2] MMA -> epilogue
  uint64_t* acc_empty = acc_full + 2;             // [2] epilogue -> MMA
  uint64_t* sums_full = acc_empty + 2;            // [2] unpack -> epilogue
  uint64_t* sums_empty = sums_full + 2;           // [2] epilogue -> unpack
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(smem + C::OFF_MISC);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(smem + C::OFF_MISC + 4);
  int* sumA = reinterpret_cast<int*>(smem + C::OFF_SUMA);   // [2][BM]
  int* sumB = reinterpret_cast<int*>(smem + C::OFF_SUMB);   // [2][BN]

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
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
    for (int i = 0; i < 2; ++i) {
      mbar_init(&acc_full[i], 1);
      mbar_init(&acc_empty[i], kEpiWarps);
      mbar_init(&sums_full[i], kConvWarps);
      mbar_init(&sums_empty[i], kEpiWarps);
    }
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
  const int per = p.num_m * p.num_n;

  if (warp == 0) {
    // ------------------------------------------------------------ TMA producer
    if (lane == 0) {
      tma_prefetch_desc(&tmA);
      tma_prefetch_desc(&tmB);
      int g = 0, issued = 0;
      bool ok = true;
      for (int t = blockIdx.x; t < p.tiles && ok; t += gridDim.x) {
        const int bz = t / per, r = t - bz * per, nb = r / p.num_m;
        const int m0 = (r - nb * p.num_m) * BM, n0 = nb * BN;
        for (int kb = 0; kb < KB; ++kb, ++g) {
          const int s = g % C::SP;
          if (!mbar_wait(&empty_p[s], ((g / C::SP) & 1) ^ 1, abort_flag, &g_gemm_err)) {
            ok = false;
            break;
          }
          uint8_t* pa = smem + C::OFF_PACK + s * C::PACK_STAGE;
          mbar_arrive_expect_tx(&full_p[s], C::PACK_STAGE);
          tma_load_3d(&tmA, &full_p[s], pa, kb * BKP, m0, bz);
          tma_load_3d(&tmB, &full_p[s], pa + C::A_PACK, kb * BKP, n0, bz);
          issued = g + 1;
        }
      }
      if (*abort_flag) {
        // Let the copies already in flight land before the CTA exits.
        for (int q = max(0, issued - C::SP); q < issued; ++q) {
          const uint32_t a = smem_u32(&full_p[q % C::SP]);
          const unsigned long long t0 = globaltimer();
          while (!mbar_try_wait(a, (q / C::SP) & 1) && globaltimer() - t0 < 100000000ull) {
          }
        }
      }
    }
  } else if (warp == 1) {
    // ------------------------------------------------------------ MMA issuer
    if (lane == 0) {
      constexpr uint32_t idesc = idesc_e4m3_f32(BM, BN);
      int g = 0, it = 0;
      bool ok = true;
      for (int t = blockIdx.x; t < p.tiles && ok; t += gridDim.x, ++it) {
        const int ab = it & 1;
        if (!mbar_wait(&acc_empty[ab], ((it >> 1) & 1) ^ 1, abort_flag, &g_gemm_err)) break;
        tc_fence_after();
        const uint32_t d = tmem_base + static_cast<uint32_t>(ab * BN);
        for (int kb = 0; kb < KB; ++kb, ++g) {
          const int s = g % C::SC;
          if (!mbar_wait(&full_c[s], (g / C::SC) & 1, abort_flag, &g_gemm_err)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t a0 = smem_u32(smem + s * C::CONV_STAGE);
          const uint32_t b0 = a0 + C::A_CONV;
#pragma unroll
          for (int k = 0; k < BK / 32; ++k)
            mma_f8f6f4(d, sw128_kmajor_desc(a0 + k * 32), sw128_kmajor_desc(b0 + k * 32), idesc,
                       (kb | k) != 0 ? 1u : 0u);
          mma_commit(&empty_c[s]);
        }
        mma_commit(&acc_full[ab]);
      }
    }
  } else if (warp < kFirstEpiWarp) {
    // ------------------------------------------------------------ unpack warps
    const int tc = threadIdx.x - kFirstConvWarp * 32;
    constexpr int NA = BM * 4 / kConvThreads, NB = BN * 4 / kConvThreads;
    int g = 0, it = 0;
    bool ok = true;
    for (int t = blockIdx.x; t < p.tiles && ok; t += gridDim.x, ++it) {
      int accA[NA], accB[NB];
#pragma unroll
      for (int j = 0; j < NA; ++j) accA[j] = 0;
#pragma unroll
      for (int j = 0; j < NB; ++j) accB[j] = 0;
      for (int kb = 0; kb < KB; ++kb, ++g) {
        const int s = g % C::SP, c = g % C::SC;
        if (!mbar_wait(&full_p[s], (g / C::SP) & 1, abort_flag, &g_gemm_err) ||
            !mbar_wait(&empty_c[c], ((g / C::SC) & 1) ^ 1, abort_flag, &g_gemm_err)) {
          ok = false;
          break;
        }
        const uint8_t* pa = smem + C::OFF_PACK + s * C::PACK_STAGE;
        const uint8_t* pb = pa + C::A_PACK;
        uint8_t* ca = smem + c * C::CONV_STAGE;
        uint8_t* cb = ca + C::A_CONV;
        uint4 va[NA], vb[NB];
#pragma unroll
        for (int j = 0; j < NA; ++j) {
          const int task = tc + j * kConvThreads;
          va[j] = *reinterpret_cast<const uint4*>(pa + (task >> 2) * BKP + (task & 3) * 16);
        }
#pragma unroll
        for (int j = 0; j < NB; ++j) {
          const int task = tc + j * kConvThreads;
          vb[j] = *reinterpret_cast<const uint4*>(pb + (task >> 2) * BKP + (task & 3) * 16);
        }
#pragma unroll
        for (int j = 0; j < NA; ++j) {
          const int task = tc + j * kConvThreads;
          accA[j] += convert_chunk(va[j], ca, task >> 2, task & 3);
        }
#pragma unroll
        for (int j = 0; j < NB; ++j) {
          const int task = tc + j * kConvThreads;
          accB[j] += convert_chunk(vb[j], cb, task >> 2, task & 3);
        }
        fence_proxy_async_smem();
        __syncwarp();
        if (lane == 0) {
          mbar_arrive(&empty_p[s]);  // packed stage consumed
          mbar_arrive(&full_c[c]);   // E4M3 stage ready for the tensor core
        }
      }
      if (!ok) break;
      // Row sums of u over the whole K for this tile: reduce the 4 threads sharing a row.
      const int ab = it & 1;
      if (!mbar_wait(&sums_empty[ab], ((it >> 1) & 1) ^ 1, abort_flag, &g_gemm_err)) break;
#pragma unroll
      for (int j = 0; j < NA; ++j) {
        int v = accA[j];
        v += __shfl_xor_sync(0xFFFFFFFFu, v, 1);
        v += __shfl_xor_sync(0xFFFFFFFFu, v, 2);
        if ((tc & 3) == 0) sumA[ab * BM + ((tc + j * kConvThreads) >> 2)] = v;
      }
#pragma unroll
      for (int j = 0; j < NB; ++j) {
        int v = accB[j];
        v += __shfl_xor_sync(0xFFFFFFFFu, v, 1);
        v += __shfl_xor_sync(0xFFFFFFFFu, v, 2);
        if ((tc & 3) == 0) sumB[ab * BN + ((tc + j * kConvThreads) >> 2)] = v;
      }
      __syncwarp();
      if (lane == 0) mbar_arrive(&sums_full[ab]);
    }
  } else {
    // ------------------------------------------------------------ epilogue warps
    const int ew = warp - kFirstEpiWarp;
    const int q = warp & 3;  // TMEM lane quarter this warp may read
    uint8_t* boxes = smem + C::OFF_STAGE + ew * 2 * C::BOX_BYTES;
    float* colv = reinterpret_cast<float*>(smem + C::OFF_SCOL) + ew * BN;  // s_b or norms of this tile
    int it = 0, nbox = 0;
    for (int t = blockIdx.x; t < p.tiles; t += gridDim.x, ++it) {
      const int bz = t / per, r = t - bz * per, nb = r / p.num_m;
      const int m0 = (r - nb * p.num_m) * BM, n0 = nb * BN;
      const int ab = it & 1;
      const uint32_t ph = (it >> 1) & 1;
      if (!mbar_wait(&acc_full[ab], ph, abort_flag, &g_gemm_err)) break;
      if (!mbar_wait(&sums_full[ab], ph, abort_flag, &g_gemm_err)) break;
      tc_fence_after();
      const int row = q * 32 + lane;
      const int m = m0 + row;
      const int corrA = 64 * p.K - 8 * sumA[ab * BM + row];
      float sa = 0.0f;
      int na = 0;
      if (m < p.M) {
        if (MODE == static_cast<int>(GemmOut::kHalf)) sa = p.s_a[m];
        if (MODE == static_cast<int>(GemmOut::kCos)) na = p.norm_a[static_cast<size_t>(bz) * p.M + m];
      }
      if (MODE != static_cast<int>(GemmOut::kS32)) {
        for (int i = lane; i < BN; i += 32) {
          const int n = n0 + i;
          float v = 0.0f;
          if (n < p.N) {
            if (MODE == static_cast<int>(GemmOut::kHalf)) v = p.s_b[n];
            else v = static_cast<float>(p.norm_b[static_cast<size_t>(bz) * p.N + n]);
          }
          colv[i] = v;
        }
        __syncwarp();
      }
#pragma unroll 1
      for (int cc = 0; cc < BN / 32; ++cc) {
        uint32_t v[32];
        tmem_ld_32x32b_x32(tmem_base + (static_cast<uint32_t>(q * 32) << 16) + ab * BN + cc * 32, v);
        tmem_ld_wait();
        if (cc == BN / 32 - 1) {
          // Accumulator and sums fully read: hand them back.
          tc_fence_before();
          __syncwarp();
          if (lane == 0) {
            mbar_arrive(&acc_empty[ab]);
          }
        }
        const int* sb = sumB + ab * BN + cc * 32;
        uint8_t* box = boxes + (nbox & 1) * C::BOX_BYTES;
        if (lane == 0) bulk_wait_group_read<1>();  // the box about to be written is free again
        __syncwarp();
        uint8_t* rowp = box + lane * (32 * C::ELEM);
        if (MODE == static_cast<int>(GemmOut::kHalf)) {
#pragma unroll
          for (int g4 = 0; g4 < 4; ++g4) {
            uint32_t w[4];
#pragma unroll
            for (int e = 0; e < 4; ++e) {
              const int i0 = g4 * 8 + 2 * e;
              const int a0 = __float2int_rn(__uint_as_float(v[i0]) * 262144.0f) + corrA - 8 * sb[i0];
              const int a1 = __float2int_rn(__uint_as_float(v[i0 + 1]) * 262144.0f) + corrA - 8 * sb[i0 + 1];
              const float y0 = __fmul_rn(__fmul_rn(static_cast<float>(a0), sa), colv[cc * 32 + i0]);
              const float y1 = __fmul_rn(__fmul_rn(static_cast<float>(a1), sa), colv[cc * 32 + i0 + 1]);
              const __half2 h = __floats2half2_rn(y0, y1);
              w[e] = *reinterpret_cast<const uint32_t*>(&h);
            }
            // 64-byte rows, 64-byte swizzle: chunk g4 of row lane
            *reinterpret_cast<uint4*>(rowp + ((g4 ^ ((lane >> 1) & 3)) << 4)) = make_uint4(w[0], w[1], w[2], w[3]);
          }
        } else {
#pragma unroll
          for (int g4 = 0; g4 < 8; ++g4) {
            uint32_t w[4];
#pragma unroll
            for (int e = 0; e < 4; ++e) {
              const int i = g4 * 4 + e;
              const int a = __float2int_rn(__uint_as_float(v[i]) * 262144.0f) + corrA - 8 * sb[i];
              if (MODE == static_cast<int>(GemmOut::kS32)) {
                w[e] = static_cast<uint32_t>(a);
              } else {
                const float nn = colv[cc * 32 + i];
                const float cs = (na == 0 || nn == 0.0f)
                                     ? 0.0f
                                     : __fdiv_rn(static_cast<float>(a),
                                                 __fsqrt_rn(__fmul_rn(static_cast<float>(na), nn)));
                w[e] = __float_as_uint(cs);
              }
            }
            // 128-byte rows, 128-byte swizzle: chunk g4 of row lane
            *reinterpret_cast<uint4*>(rowp + ((g4 ^ (lane & 7)) << 4)) = make_uint4(w[0], w[1], w[2], w[3]);
          }
        }
        fence_proxy_async_smem();
        __syncwarp();
        if (lane == 0) {
          tma_store_3d(&tmD, box, n0 + cc * 32, m0 + q * 32, bz);
          bulk_commit_group();
        }
        ++nbox;
      }
      __syncwarp();
      if (lane == 0) mbar_arrive(&sums_empty[ab]);
    }
    if (lane == 0) bulk_wait_group_all();
    __syncwarp();
  }

  // Teardown: every MMA must have completed before TMEM is released.
  if (warp == 1 && lane == 0 && *abort_flag) {
    for (int i = 0; i < 2; ++i) {
      const unsigned long long t0 = globaltimer();
      const uint32_t a = smem_u32(&acc_full[i]);
      while (!mbar_try_wait(a, 0) && !mbar_try_wait(a, 1) && globaltimer() - t0 < 100000000ull) {
      }
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
bool make_operand_map(CUtensorMap* map, const uint8_t* base, int K, int rows, int batch,
                      long long batch_stride_rows, int box_rows) {
  auto enc = get_encode_fn();
  if (!enc) return false;
  const cuuint64_t kb = static_cast<cuuint64_t>(K / 2);
  cuuint64_t dims[3] = {kb, static_cast<cuuint64_t>(rows), static_cast<cuuint64_t>(batch)};
  const long long bs = batch_stride_rows > 0 ? batch_stride_rows : rows;
  cuuint64_t strides[2] = {kb, static_cast<cuuint64_t>(bs) * kb};
  cuuint32_t box[3] = {static_cast<cuuint32_t>(BKP), static_cast<cuuint32_t>(box_rows), 1};
  cuuint32_t estr[3] = {1, 1, 1};
  return enc(map, CU_TENSOR_MAP_DATA_TYPE_UINT8, 3, const_cast<uint8_t*>(base), dims, strides, box, estr,
             CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_NONE, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
             CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// 3-D map over the output [batch][rows][cols] with row pitch `pitch` elements;
// 32 x 32 boxes in the swizzle the epilogue writes.
bool make_output_map(CUtensorMap* map, void* base, GemmOut out, int rows, int cols, int pitch, int batch) {
  auto enc = get_encode_fn();
  if (!enc) return false;
  const int es = (out == GemmOut::kHalf) ? 2 : 4;
  const CUtensorMapDataType dt = (out == GemmOut::kHalf)  ? CU_TENSOR_MAP_DATA_TYPE_FLOAT16
                                 : (out == GemmOut::kS32) ? CU_TENSOR_MAP_DATA_TYPE_INT32
                                                          : CU_TENSOR_MAP_DATA_TYPE_FLOAT32;
  cuuint64_t dims[3] = {static_cast<cuuint64_t>(cols), static_cast<cuuint64_t>(rows), static_cast<cuuint64_t>(batch)};
  cuuint64_t strides[2] = {static_cast<cuuint64_t>(pitch) * es, static_cast<cuuint64_t>(pitch) * es * rows};
  cuuint32_t box[3] = {32, 32, 1};
  cuuint32_t estr[3] = {1, 1, 1};
  return enc(map, dt, 3, base, dims, strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE,
             es == 2 ? CU_TENSOR_MAP_SWIZZLE_64B : CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_NONE,
             CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

int num_sms() {
  static int n = 0;
  if (n == 0) {
    int dev = 0;
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev);
    if (n <= 0) n = 1;
  }
  return n;
}

template <int BN, int MODE>
cudaError_t launch_cfg(const GemmArgs& g, cudaStream_t stream) {
  using C = Cfg<BN, MODE>;
  static bool attr_set = false;
  if (!attr_set) {
    cudaError_t e =
        cudaFuncSetAttribute(w4a4_gemm_kernel<BN, MODE>, cudaFuncAttributeMaxDynamicSharedMemorySize, C::SMEM);
    if (e != cudaSuccess) return e;
    attr_set = true;
  }
  CUtensorMap ma, mb, md;
  if (!make_operand_map(&ma, g.A, g.K, g.M, g.batch, g.a_batch_stride, BM)) return cudaErrorInvalidValue;
  if (!make_operand_map(&mb, g.B, g.K, g.N, g.batch, g.b_batch_stride, BN)) return cudaErrorInvalidValue;
  const int pitch = g.d_pitch > 0 ? g.d_pitch : g.N;
  if (!make_output_map(&md, g.D, g.out, g.M, g.N, pitch, g.batch)) return cudaErrorInvalidValue;
  Params p;
  p.M = g.M;
  p.N = g.N;
  p.K = g.K;
  p.batch = g.batch;
  p.num_m = (g.M + BM - 1) / BM;
  p.num_n = (g.N + BN - 1) / BN;
  p.tiles = p.num_m * p.num_n * g.batch;
  p.s_a = g.s_a;
  p.s_b = g.s_b;
  p.norm_a = g.norm_a;
  p.norm_b = g.norm_b;
  const int grid = p.tiles < num_sms() ? p.tiles : num_sms();
  w4a4_gemm_kernel<BN, MODE><<<grid, kThreads, C::SMEM, stream>>>(ma, mb, md, p);
  return cudaGetLastError();
}

}  // namespace

cudaError_t launch_w4a4_gemm(const GemmArgs& g, cudaStream_t stream) {
  if (g.M <= 0 || g.N <= 0 || g.batch <= 0) return cudaSuccess;
  switch (g.out) {
    case GemmOut::kHalf:
      return (g.N >= 1024) ? launch_cfg<256, 0>(g, stream) : launch_cfg<128, 0>(g, stream);
    case GemmOut::kS32:
      return launch_cfg<128, 1>(g, stream);
    case GemmOut::kCos:
      return launch_cfg<128, 2>(g, stream);
  }
  return cudaErrorInvalidValue;
}

unsigned int gemm_read_and_clear_error() {
  unsigned int v = 0, z = 0;
  cudaMemcpyFromSymbol(&v, g_gemm_err, sizeof(v));
  cudaMemcpyToSymbol(g_gemm_err, &z, sizeof(z));
  return v;
}

}  // namespace p4q
