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
//   warp 0       MMA: 4 x tcgen05.mma (K = 32 each) per 128-deep k-block into
//                one of two TMEM accumulators (128 lanes x BN fp32 columns);
//   warps 1-8    unpack: 16-byte global loads of the packed A and B rows of the
//                next k-blocks into registers (three k-blocks in flight, the
//                tiles prefetched into L2 by TMA further ahead), then the E4M3
//                bytes written in the 128-byte swizzled K-major layout the
//                tensor core reads (ring of SC stages), plus the per-row sums of
//                u for the correction;
//   warps 9-12   epilogue of the previous tile, overlapped with the next
//                tile's main loop: tcgen05.ld, correction, scaling, a 32 x 32
//                box staged in swizzled shared memory, TMA store.
// Loading the packed operands straight into registers keeps the only shared
// memory traffic of the main loop to the E4M3 stores and the tensor core's
// operand reads.
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
constexpr int kGroups = 2;                   // unpack groups, each converts every kGroups-th k-block
constexpr int kGroupWarps = 8;
constexpr int kConvWarps = kGroups * kGroupWarps;
constexpr int kEpiWarps = 4;
constexpr int kGroupThreads = kGroupWarps * 32;
constexpr int kRowStep = kGroupThreads / 4;  // rows between the chunks one unpack thread handles
constexpr int kFirstConvWarp = 1;
constexpr int kFirstEpiWarp = kFirstConvWarp + kConvWarps;
constexpr int kThreads = (kFirstEpiWarp + kEpiWarps) * 32;
constexpr int kPrefetchAhead = 6;
#ifndef P4Q_UNPACK_DEPTH
#define P4Q_UNPACK_DEPTH 1
#endif
constexpr int kDepth = P4Q_UNPACK_DEPTH;       // k-blocks of one group held in registers (1 or 2)            // k-blocks prefetched into L2 ahead of the loads

template <int BN, int MODE>
struct Cfg {
  static constexpr int A_CONV = BM * BK;
  static constexpr int B_CONV = BN * BK;
  static constexpr int CONV_STAGE = A_CONV + B_CONV;
  static constexpr int ELEM = (MODE == static_cast<int>(GemmOut::kHalf)) ? 2 : 4;
  static constexpr int BOX_BYTES = 32 * 32 * ELEM;  // one 32 x 32 output box
  static constexpr int FIXED = kEpiWarps * 2 * BOX_BYTES + 2 * kGroups * (BM + BN) * 4 + 2 * BN * 4 + 512;
  static constexpr int SC_FIT = (232448 - 1024 - FIXED) / CONV_STAGE > 8 ? 8 : (232448 - 1024 - FIXED) / CONV_STAGE;
  // Every stage must belong to one unpack group (SC % kGroups == 0): a group
  // then reuses a stage only after its own previous use of it, so its parity
  // wait on the stage's barrier can never run more than one phase ahead.
  static constexpr int SC = SC_FIT - SC_FIT % kGroups;
  static constexpr int OFF_STAGE = SC * CONV_STAGE;                // epilogue boxes, 2 per warp
  static constexpr int OFF_SUMA = OFF_STAGE + kEpiWarps * 2 * BOX_BYTES;
  static constexpr int OFF_SUMB = OFF_SUMA + 2 * kGroups * BM * 4;
  static constexpr int OFF_SCOL = OFF_SUMB + 2 * kGroups * BN * 4;  // column scale / norm and -8 sum_u caches
  static constexpr int OFF_BAR = OFF_SCOL + 2 * BN * 4;
  static constexpr int NBAR = 2 * SC + 8;
  static constexpr int OFF_MISC = OFF_BAR + NBAR * 8;
  static constexpr int SMEM = 1024 + OFF_MISC + 16;
  static constexpr uint32_t TMEM_COLS = 2 * BN;
  static_assert(SC >= 2 && SC % kGroups == 0, "E4M3 stages: at least two, a multiple of the groups");
  static_assert(SMEM <= 232448, "shared memory budget");
};

struct Params {
  const uint8_t* A;  // [batch][M][K/2] packed, batch stride a_bs rows
  const uint8_t* B;  // [batch][N][K/2]
  long long a_bs, b_bs;
  int M, N, K, batch;
  int num_m, num_n, tiles;
  const float* s_a;
  const float* s_b;
  const int32_t* norm_a;
  const int32_t* norm_b;
};

// Named barrier among the epilogue warps only (id 1).
__device__ __forceinline__ void epi_sync() {
  asm volatile("bar.sync 1, %0;" ::"n"(kEpiWarps * 32) : "memory");
}

// Offset codes u = v + 8 of the even (lo) and odd (hi) nibbles of a packed
// word, one per byte. The shift by 4 is done as a high multiply so that it
// runs on the FMA pipe rather than the integer-logic pipe.
__device__ __forceinline__ uint32_t nib_lo(uint32_t w) { return (w & 0x0F0F0F0Fu) ^ 0x08080808u; }
__device__ __forceinline__ uint32_t nib_hi(uint32_t w) {
  return (__umulhi(w, 0x10000000u) & 0x0F0F0F0Fu) ^ 0x08080808u;
}

// Writes the 32 E4M3 bytes of one 16-byte packed chunk (32 codes of one row)
// at logical byte offset 32*c of row r of a 128-byte-swizzled K-major tile and
// adds the sum of the 32 offset codes u to acc (dp4a, FMA pipe).
__device__ __forceinline__ void convert_chunk(const uint4 p, uint8_t* conv_tile, int r, int c, uint32_t& acc) {
  const uint32_t l0 = nib_lo(p.x), h0 = nib_hi(p.x), l1 = nib_lo(p.y), h1 = nib_hi(p.y);
  const uint32_t l2 = nib_lo(p.z), h2 = nib_hi(p.z), l3 = nib_lo(p.w), h3 = nib_hi(p.w);
  uint8_t* row = conv_tile + r * 128;
  const int sw = r & 7;
  *reinterpret_cast<uint4*>(row + (((2 * c) ^ sw) << 4)) = make_uint4(l0, h0, l1, h1);
  *reinterpret_cast<uint4*>(row + (((2 * c + 1) ^ sw) << 4)) = make_uint4(l2, h2, l3, h3);
  constexpr uint32_t ones = 0x01010101u;
  acc = __dp4a(l0, ones, acc);
  acc = __dp4a(h0, ones, acc);
  acc = __dp4a(l1, ones, acc);
  acc = __dp4a(h1, ones, acc);
  acc = __dp4a(l2, ones, acc);
  acc = __dp4a(h2, ones, acc);
  acc = __dp4a(l3, ones, acc);
  acc = __dp4a(h3, ones, acc);
}

// The two halves of convert_chunk, so that the unpack can run before the
// wait for a free stage and only the stores after it.
struct Unpacked {
  uint4 lo, hi;  // E4M3 bytes of the 32 codes, in the order convert_chunk stores them
};

__device__ __forceinline__ Unpacked unpack_chunk(const uint4 p, uint32_t& acc) {
  Unpacked u;
  u.lo = make_uint4(nib_lo(p.x), nib_hi(p.x), nib_lo(p.y), nib_hi(p.y));
  u.hi = make_uint4(nib_lo(p.z), nib_hi(p.z), nib_lo(p.w), nib_hi(p.w));
  constexpr uint32_t ones = 0x01010101u;
  acc = __dp4a(u.lo.x, ones, acc);
  acc = __dp4a(u.lo.y, ones, acc);
  acc = __dp4a(u.lo.z, ones, acc);
  acc = __dp4a(u.lo.w, ones, acc);
  acc = __dp4a(u.hi.x, ones, acc);
  acc = __dp4a(u.hi.y, ones, acc);
  acc = __dp4a(u.hi.z, ones, acc);
  acc = __dp4a(u.hi.w, ones, acc);
  return u;
}

__device__ __forceinline__ void store_chunk(const Unpacked& u, uint8_t* conv_tile, int r, int c) {
  uint8_t* row = conv_tile + r * 128;
  const int sw = r & 7;
  *reinterpret_cast<uint4*>(row + (((2 * c) ^ sw) << 4)) = u.lo;
  *reinterpret_cast<uint4*>(row + (((2 * c + 1) ^ sw) << 4)) = u.hi;
}

template <int BN, int MODE>
__global__ void __launch_bounds__(kThreads, 1)
    w4a4_gemm_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB,
                     const __grid_constant__ CUtensorMap tmD, const Params p) {
  using C = Cfg<BN, MODE>;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + C::OFF_BAR);
  uint64_t* full_c = bars;                        // unpack -> MMA
  uint64_t* empty_c = full_c + C::SC;             // MMA -> unpack
  uint64_t* acc_full = empty_c + C::SC;           // [2] MMA -> epilogue
  uint64_t* acc_empty = acc_full + 2;             // [2] epilogue -> MMA
  uint64_t* sums_full = acc_empty + 2;            // [2] unpack -> epilogue
  uint64_t* sums_empty = sums_full + 2;           // [2] epilogue -> unpack
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(smem + C::OFF_MISC);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(smem + C::OFF_MISC + 4);
  int* sumA = reinterpret_cast<int*>(smem + C::OFF_SUMA);   // [2][kGroups][BM] partial sums per group
  int* sumB = reinterpret_cast<int*>(smem + C::OFF_SUMB);   // [2][kGroups][BN]

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int KB = p.K / BK;

  if (threadIdx.x == 0) {
    for (int i = 0; i < C::SC; ++i) {
      mbar_init(&full_c[i], kGroupWarps);
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
  if (warp == 0) {
    tmem_alloc(tmem_slot, C::TMEM_COLS);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem_base = *tmem_slot;
  pdl_wait();  // operands and scales come from the previous kernel
  pdl_launch_dependents();
  const int per = p.num_m * p.num_n;

  if (warp == 0) {
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
    // Group grp converts the k-blocks g with g % kGroups == grp (g counts the
    // k-blocks of all tiles this CTA processes), so kGroups independent
    // load -> convert -> store chains are in flight at once.
    const int cw = warp - kFirstConvWarp;
    const int grp = cw / kGroupWarps;
    const int tc = threadIdx.x - (kFirstConvWarp + grp * kGroupWarps) * 32;
    constexpr int NA = BM * 4 / kGroupThreads, NB = BN * 4 / kGroupThreads, NT = NA + NB;
    const int rbase = tc >> 2, chunk = tc & 3;
    const size_t rowbytes = static_cast<size_t>(p.K) >> 1;
    const bool prefetcher = (tc == 0);
    if (prefetcher) {
      tma_prefetch_desc(&tmA);
      tma_prefetch_desc(&tmB);
    }
    int gbase = 0, it = 0;  // gbase: global index of the tile's first k-block
    bool ok = true;
    for (int t = blockIdx.x; t < p.tiles && ok; t += gridDim.x, ++it, gbase += KB) {
      const int bz = t / per, r = t - bz * per, nb = r / p.num_m;
      const int m0 = (r - nb * p.num_m) * BM, n0 = nb * BN;
      // This thread's rows: rbase + kRowStep * j of the A and B tiles; rows
      // outside the matrix read as zero codes.
      const uint8_t* baseA = p.A + (static_cast<size_t>(bz) * p.a_bs + m0 + rbase) * rowbytes + chunk * 16;
      const uint8_t* baseB = p.B + (static_cast<size_t>(bz) * p.b_bs + n0 + rbase) * rowbytes + chunk * 16;
      const size_t step = static_cast<size_t>(kRowStep) * rowbytes;
      uint32_t valid = 0;
#pragma unroll
      for (int j = 0; j < NA; ++j) valid |= (m0 + rbase + kRowStep * j < p.M) ? (1u << j) : 0u;
#pragma unroll
      for (int j = 0; j < NB; ++j) valid |= (n0 + rbase + kRowStep * j < p.N) ? (1u << (NA + j)) : 0u;
      // first k-block of this tile that belongs to this group
      const int kb0 = ((grp - gbase) % kGroups + kGroups) % kGroups;
      if (prefetcher && grp == 0) {
        for (int kb = 0; kb < min(KB, kPrefetchAhead); ++kb) {
          tma_prefetch_l2_3d(&tmA, kb * BKP, m0, bz);
          tma_prefetch_l2_3d(&tmB, kb * BKP, n0, bz);
        }
      }
      uint32_t accA[NA], accB[NB];
#pragma unroll
      for (int j = 0; j < NA; ++j) accA[j] = 0;
#pragma unroll
      for (int j = 0; j < NB; ++j) accB[j] = 0;
      uint4 buf[kDepth][NT];
      auto load = [&](uint4 (&v)[NT], int kb) {
        const size_t off = static_cast<size_t>(kb) * BKP;
#pragma unroll
        for (int j = 0; j < NA; ++j)
          v[j] = (valid >> j) & 1u ? ldg_stream16(baseA + j * step + off) : make_uint4(0u, 0u, 0u, 0u);
#pragma unroll
        for (int j = 0; j < NB; ++j)
          v[NA + j] = (valid >> (NA + j)) & 1u ? ldg_stream16(baseB + j * step + off) : make_uint4(0u, 0u, 0u, 0u);
      };
      auto convert = [&](const uint4 (&v)[NT], int kb) -> bool {
        const int g = gbase + kb;
        const int c = g % C::SC;
        if (prefetcher && grp == 0) {
          for (int q = kb + kPrefetchAhead; q < min(KB, kb + kPrefetchAhead + kGroups); ++q) {
            tma_prefetch_l2_3d(&tmA, q * BKP, m0, bz);
            tma_prefetch_l2_3d(&tmB, q * BKP, n0, bz);
          }
        }
        if (!mbar_wait_warp(&empty_c[c], ((g / C::SC) & 1) ^ 1, abort_flag, &g_gemm_err)) return false;
        uint8_t* ca = smem + c * C::CONV_STAGE;
        uint8_t* cb = ca + C::A_CONV;
#pragma unroll
        for (int j = 0; j < NA; ++j) convert_chunk(v[j], ca, rbase + kRowStep * j, chunk, accA[j]);
#pragma unroll
        for (int j = 0; j < NB; ++j) convert_chunk(v[NA + j], cb, rbase + kRowStep * j, chunk, accB[j]);
        fence_proxy_async_smem();
        __syncwarp();
        if (lane == 0) mbar_arrive(&full_c[c]);  // E4M3 stage ready for the tensor core
        return true;
      };
      if constexpr (kDepth == 1) {
        // One k-block of this group in flight: the next load is issued as soon
        // as the registers are free, a whole group period ahead of its use.
        if (kb0 < KB) load(buf[0], kb0);
        for (int kb = kb0; kb < KB && ok; kb += kGroups) {
          ok = convert(buf[0], kb);
          if (ok && kb + kGroups < KB) load(buf[0], kb + kGroups);
        }
      } else {
        // Two of this group's k-blocks in flight in registers.
        if (kb0 < KB) load(buf[0], kb0);
        if (kb0 + kGroups < KB) load(buf[kDepth - 1], kb0 + kGroups);
        for (int kb = kb0; kb < KB && ok; kb += 2 * kGroups) {
          ok = convert(buf[0], kb);
          if (!ok || kb + kGroups >= KB) break;
          if (kb + 2 * kGroups < KB) load(buf[0], kb + 2 * kGroups);
          ok = convert(buf[kDepth - 1], kb + kGroups);
          if (!ok) break;
          if (kb + 3 * kGroups < KB) load(buf[kDepth - 1], kb + 3 * kGroups);
        }
      }
      if (!ok) break;
      // This group's row sums of u for the tile: reduce the 4 threads sharing a row.
      const int ab = it & 1;
      if (!mbar_wait_warp(&sums_empty[ab], ((it >> 1) & 1) ^ 1, abort_flag, &g_gemm_err)) break;
#pragma unroll
      for (int j = 0; j < NA; ++j) {
        int v = static_cast<int>(accA[j]);
        v += __shfl_xor_sync(0xFFFFFFFFu, v, 1);
        v += __shfl_xor_sync(0xFFFFFFFFu, v, 2);
        if (chunk == 0) sumA[(ab * kGroups + grp) * BM + rbase + kRowStep * j] = v;
      }
#pragma unroll
      for (int j = 0; j < NB; ++j) {
        int v = static_cast<int>(accB[j]);
        v += __shfl_xor_sync(0xFFFFFFFFu, v, 1);
        v += __shfl_xor_sync(0xFFFFFFFFu, v, 2);
        if (chunk == 0) sumB[(ab * kGroups + grp) * BN + rbase + kRowStep * j] = v;
      }
      __syncwarp();
      if (lane == 0) mbar_arrive(&sums_full[ab]);
    }
  } else {
    // ------------------------------------------------------------ epilogue warps
    const int ew = warp - kFirstEpiWarp;
    const int q = warp & 3;  // TMEM lane quarter this warp may read
    uint8_t* boxes = smem + C::OFF_STAGE + ew * 2 * C::BOX_BYTES;
    float* colv = reinterpret_cast<float*>(smem + C::OFF_SCOL);  // s_b or norms of this tile
    // The epilogue warps synchronize among themselves with a named barrier, so
    // they all run the same number of iterations: after a failed wait a warp
    // keeps looping (doing no work) instead of leaving the others at the barrier.
    int it = 0, nbox = 0;
    bool failed = false;
    for (int t = blockIdx.x; t < p.tiles; t += gridDim.x, ++it) {
      const int bz = t / per, r = t - bz * per, nb = r / p.num_m;
      const int m0 = (r - nb * p.num_m) * BM, n0 = nb * BN;
      const int ab = it & 1;
      const uint32_t ph = (it >> 1) & 1;
      if (!failed && !(mbar_wait_warp(&acc_full[ab], ph, abort_flag, &g_gemm_err) &&
                       mbar_wait_warp(&sums_full[ab], ph, abort_flag, &g_gemm_err)))
        failed = true;
      tc_fence_after();
      const int row = q * 32 + lane;
      const int m = m0 + row;
      // -8 * (column sums of u of the B rows of this tile), all groups combined
      float* sbw = reinterpret_cast<float*>(smem + C::OFF_SCOL) + BN;
      epi_sync();  // every epilogue warp is done with the previous tile's caches
      if (!failed) {
        for (int i = ew * 32 + lane; i < BN; i += kEpiWarps * 32) {
          int v = 0;
#pragma unroll
          for (int q2 = 0; q2 < kGroups; ++q2) v += sumB[(ab * kGroups + q2) * BN + i];
          sbw[i] = static_cast<float>(-8 * v);
          if (MODE != static_cast<int>(GemmOut::kS32)) {
            const int n = n0 + i;
            float cv = 0.0f;
            if (n < p.N) {
              if (MODE == static_cast<int>(GemmOut::kHalf)) cv = p.s_b[n];
              else cv = static_cast<float>(p.norm_b[static_cast<size_t>(bz) * p.N + n]);
            }
            colv[i] = cv;
          }
        }
      }
      epi_sync();  // caches of this tile complete
      if (failed) continue;
      int sa_u = 0;
#pragma unroll
      for (int q2 = 0; q2 < kGroups; ++q2) sa_u += sumA[(ab * kGroups + q2) * BM + row];
      // acc = P - 8 sum_k u_a - 8 sum_k u_b + 64 K, evaluated in fp32: every
      // term and partial result is an integer of magnitude < 2^24, so the
      // fused multiply-add below is exact.
      const float corrA = static_cast<float>(64 * p.K - 8 * sa_u);
      float sa = 0.0f;
      int na = 0;
      if (m < p.M) {
        if (MODE == static_cast<int>(GemmOut::kHalf)) sa = p.s_a[m];
        if (MODE == static_cast<int>(GemmOut::kCos)) na = p.norm_a[static_cast<size_t>(bz) * p.M + m];
      }
#pragma unroll 1
      for (int cc = 0; cc < BN / 32; ++cc) {
        uint8_t* box = boxes + (nbox & 1) * C::BOX_BYTES;
        if (lane == 0) bulk_wait_group_read<1>();  // the box about to be written is free again
        __syncwarp();
        uint8_t* rowp = box + lane * (32 * C::ELEM);
#pragma unroll 1
        for (int h = 0; h < 2; ++h) {
          const int c0 = cc * 32 + h * 16;  // first of the 16 columns of this half
          uint32_t v[16];
          tmem_ld_32x32b_x16(tmem_base + (static_cast<uint32_t>(q * 32) << 16) + ab * BN + c0, v);
          tmem_ld_wait();
          if (cc == BN / 32 - 1 && h == 1) {
            // Accumulator fully read: hand it back to the MMA warp.
            tc_fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive(&acc_empty[ab]);
          }
          float acc[16];  // exact integers
#pragma unroll
          for (int i = 0; i < 16; ++i)
            acc[i] = __fmaf_rn(__uint_as_float(v[i]), 262144.0f, corrA + sbw[c0 + i]);
          if (MODE == static_cast<int>(GemmOut::kHalf)) {
#pragma unroll
            for (int g2 = 0; g2 < 2; ++g2) {
              uint32_t w[4];
#pragma unroll
              for (int e = 0; e < 4; ++e) {
                const int i0 = g2 * 8 + 2 * e;
                const float y0 = __fmul_rn(__fmul_rn(acc[i0], sa), colv[c0 + i0]);
                const float y1 = __fmul_rn(__fmul_rn(acc[i0 + 1], sa), colv[c0 + i0 + 1]);
                const __half2 hh = __floats2half2_rn(y0, y1);
                w[e] = *reinterpret_cast<const uint32_t*>(&hh);
              }
              // 64-byte rows, 64-byte swizzle: 16-byte chunk (2h + g2) of row `lane`
              const int ch = 2 * h + g2;
              *reinterpret_cast<uint4*>(rowp + ((ch ^ ((lane >> 1) & 3)) << 4)) = make_uint4(w[0], w[1], w[2], w[3]);
            }
          } else {
#pragma unroll
            for (int g4 = 0; g4 < 4; ++g4) {
              uint32_t w[4];
#pragma unroll
              for (int e = 0; e < 4; ++e) {
                const int i = g4 * 4 + e;
                if (MODE == static_cast<int>(GemmOut::kS32)) {
                  w[e] = static_cast<uint32_t>(__float2int_rn(acc[i]));
                } else {
                  const float nn = colv[c0 + i];
                  const float cs = (na == 0 || nn == 0.0f)
                                       ? 0.0f
                                       : __fdiv_rn(acc[i],
                                                   __fsqrt_rn(__fmul_rn(static_cast<float>(na), nn)));
                  w[e] = __float_as_uint(cs);
                }
              }
              // 128-byte rows, 128-byte swizzle: 16-byte chunk (4h + g4) of row `lane`
              const int ch = 4 * h + g4;
              *reinterpret_cast<uint4*>(rowp + ((ch ^ (lane & 7)) << 4)) = make_uint4(w[0], w[1], w[2], w[3]);
            }
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
  if (warp == 0 && lane == 0 && *abort_flag) {
    for (int i = 0; i < 2; ++i) {
      const unsigned long long t0 = globaltimer();
      const uint32_t a = smem_u32(&acc_full[i]);
      while (!mbar_try_wait(a, 0) && !mbar_try_wait(a, 1) && globaltimer() - t0 < 100000000ull) {
      }
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 0) {
    tc_fence_after();
    tmem_dealloc(tmem_base, C::TMEM_COLS);
  }
}

// ============================================================================
// CTA-pair variant (tcgen05 cta_group::2): a cluster of two CTAs computes a
// 256 x 256 output tile. CTA r of the pair unpacks rows 128r..128r+127 of the
// A tile and of the B tile into its own shared memory; the leader (r = 0)
// issues M = 256 MMAs that read both CTAs' operands, and each CTA's TMEM
// receives its 128 rows of the accumulator. Per SM this halves the B rows
// unpacked per multiply-accumulate compared with a 128 x 256 tile of one CTA.
// The per-row sums of u of the B tile are exchanged between the two CTAs
// through distributed shared memory.
// ============================================================================
namespace pair {

// Pipeline shape of the pair kernel (compile-time; the defaults measured
// best on GB300): unpack groups (each converts every kGroups-th k-block),
// packed TMA stages, and the k-blocks prefetched into L2 ahead of them.
#ifndef P4Q_PAIR_GROUPS
#define P4Q_PAIR_GROUPS 2
#endif
#ifndef P4Q_PAIR_PACK
#define P4Q_PAIR_PACK 4
#endif
#ifndef P4Q_PAIR_SPIN
#define P4Q_PAIR_SPIN 2
#endif
#if P4Q_PAIR_SPIN & 1
#define PAIR_WAIT_MMA mbar_wait_spin
#else
#define PAIR_WAIT_MMA mbar_wait
#endif
#if P4Q_PAIR_SPIN & 2
#define PAIR_WAIT_CONV mbar_wait_spin_warp
#else
#define PAIR_WAIT_CONV mbar_wait_warp
#endif
#ifndef P4Q_PAIR_PREFETCH
#define P4Q_PAIR_PREFETCH 6
#endif
constexpr int kPrefetchAhead = P4Q_PAIR_PREFETCH;  // k-blocks prefetched into L2 ahead of the TMA loads
constexpr int kGroups = P4Q_PAIR_GROUPS;
constexpr int kGroupWarps = kConvWarps / kGroups;
constexpr int kGroupThreads = kGroupWarps * 32;
constexpr int kRowStep = kGroupThreads / 4;

constexpr int BN = 256;      // output columns per pair
constexpr int HB = BN / 2;   // B rows unpacked per CTA
constexpr int A_CONV = BM * BK;
constexpr int B_CONV = HB * BK;
constexpr int CONV_STAGE = A_CONV + B_CONV;
constexpr uint32_t TMEM_COLS = 2 * BN;

constexpr int A_PACK = BM * BKP;            // packed A bytes per k-block (this CTA's rows)
constexpr int PACK_STAGE = A_PACK + HB * BKP;  // packed A + B bytes per k-block
constexpr int kProducerWarp = kFirstEpiWarp + kEpiWarps;
constexpr int kPairThreads = (kProducerWarp + 1) * 32;

template <int MODE>  // GemmOut::kHalf or kS32
struct Lay {
  static constexpr int ELEM = (MODE == static_cast<int>(GemmOut::kHalf)) ? 2 : 4;
  static constexpr int BOX_BYTES = 32 * 32 * ELEM;  // one 32 x 32 output box
  // packed stages: a multiple of the unpack groups, so that each belongs to one group
  static constexpr int P = (MODE == static_cast<int>(GemmOut::kHalf)) ? P4Q_PAIR_PACK : 2;
  static constexpr int FIXED = kEpiWarps * 2 * BOX_BYTES + 2 * kGroups * (BM + BN) * 4 + 2 * BN * 4 + 512;
  static constexpr int SC_ROOM = (232448 - 1024 - FIXED - P * PACK_STAGE) / CONV_STAGE;
  static constexpr int SC_FIT = SC_ROOM > 8 ? 8 : SC_ROOM;
  static constexpr int SC = SC_FIT - SC_FIT % kGroups;
  static constexpr int OFF_PACK = SC * CONV_STAGE;
  static constexpr int OFF_STAGE = OFF_PACK + P * PACK_STAGE;
  static constexpr int OFF_SUMA = OFF_STAGE + kEpiWarps * 2 * BOX_BYTES;
  static constexpr int OFF_SUMB = OFF_SUMA + 2 * kGroups * BM * 4;
  static constexpr int OFF_SCOL = OFF_SUMB + 2 * kGroups * BN * 4;
  static constexpr int OFF_BAR = OFF_SCOL + 2 * BN * 4;
  static constexpr int NBAR = 2 * SC + 8 + 2 * P;
  static constexpr int OFF_MISC = OFF_BAR + NBAR * 8;
  static constexpr int SMEM = 1024 + OFF_MISC + 16;
  static_assert(SC >= 2 && SC % kGroups == 0, "E4M3 stages");
  static_assert(P >= 2 && P % kGroups == 0, "packed stages");
  static_assert(SMEM <= 232448, "shared memory budget");
};

template <int MODE>
__global__ void __cluster_dims__(2, 1, 1) __launch_bounds__(kPairThreads, 1)
    w4a4_gemm_pair_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB,
                          const __grid_constant__ CUtensorMap tmD, const Params p) {
  using L = Lay<MODE>;
  constexpr int SC = L::SC, P = L::P, BOX_BYTES = L::BOX_BYTES, OFF_STAGE = L::OFF_STAGE, OFF_SUMA = L::OFF_SUMA,
                OFF_SUMB = L::OFF_SUMB, OFF_SCOL = L::OFF_SCOL, OFF_BAR = L::OFF_BAR, OFF_MISC = L::OFF_MISC;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + OFF_BAR);
  uint64_t* full_c = bars;              // [SC] leader: both CTAs' unpack -> MMA
  uint64_t* empty_c = full_c + SC;      // [SC] MMA commit (both CTAs) -> unpack
  uint64_t* acc_full = empty_c + SC;    // [2] MMA commit (both CTAs) -> epilogue
  uint64_t* acc_empty = acc_full + 2;   // [2] leader: both CTAs' epilogues -> MMA
  uint64_t* sums_full = acc_empty + 2;  // [2] both CTAs' unpack -> epilogue
  uint64_t* sums_empty = sums_full + 2; // [2] both CTAs' epilogues -> unpack
  uint64_t* pack_full = sums_empty + 2; // [P] TMA of the packed operands -> unpack
  uint64_t* pack_empty = pack_full + P; // [P] unpack (this CTA) -> producer
  uint8_t* pack = smem + L::OFF_PACK;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(smem + OFF_MISC);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(smem + OFF_MISC + 4);
  int* sumA = reinterpret_cast<int*>(smem + OFF_SUMA);  // [2][kGroups][BM]
  int* sumB = reinterpret_cast<int*>(smem + OFF_SUMB);  // [2][kGroups][BN], both halves
  float* colv = reinterpret_cast<float*>(smem + OFF_SCOL);
  float* sbw = colv + BN;

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const uint32_t rank = cluster_ctarank(), peer = rank ^ 1u;
  const int KB = p.K / BK;
  const int per = p.num_m * p.num_n;  // pair tiles per batch (num_m counts 256-row tiles)

  if (threadIdx.x == 0) {
    for (int i = 0; i < SC; ++i) {
      mbar_init(&full_c[i], 2 * kGroupWarps);  // the unpack warps of both CTAs
      mbar_init(&empty_c[i], 1);
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(&acc_full[i], 1);
      mbar_init(&acc_empty[i], 2 * kEpiWarps);
      mbar_init(&sums_full[i], 2 * kConvWarps);
      mbar_init(&sums_empty[i], 2 * kEpiWarps);
    }
    for (int i = 0; i < P; ++i) {
      mbar_init(&pack_full[i], 1);
      mbar_init(&pack_empty[i], kGroupWarps);  // the unpack warps of the stage's group
    }
    *abort_flag = 0;
    fence_barrier_init();
  }
  if (warp == 0) {
    tmem_alloc_pair(tmem_slot, TMEM_COLS);
    tmem_relinquish_pair();
  }
  tc_fence_before();
  cluster_sync();  // barriers of both CTAs initialized, TMEM allocated in both
  tc_fence_after();
  const uint32_t tmem_base = *tmem_slot;
  pdl_wait();  // operands and scales come from the previous kernel
  pdl_launch_dependents();

  if (warp == 0) {
    // ------------------------------------------------------------ MMA issuer (leader)
    if (lane == 0 && rank == 0) {
      constexpr uint32_t idesc = idesc_e4m3_f32(2 * BM, BN);
      int g = 0, it = 0;
      bool ok = true;
      for (int t = cluster_id_x(); t < p.tiles && ok; t += nclusters_x(), ++it) {
        const int ab = it & 1;
        if (!mbar_wait(&acc_empty[ab], ((it >> 1) & 1) ^ 1, abort_flag, &g_gemm_err)) break;
        tc_fence_after();
        const uint32_t d = tmem_base + static_cast<uint32_t>(ab * BN);
        for (int kb = 0; kb < KB; ++kb, ++g) {
          const int s = g % SC;
          if (!PAIR_WAIT_MMA(&full_c[s], (g / SC) & 1, abort_flag, &g_gemm_err)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t a0 = smem_u32(smem + s * CONV_STAGE);
          const uint32_t b0 = a0 + A_CONV;
#pragma unroll
          for (int k = 0; k < BK / 32; ++k)
            mma_f8f6f4_pair(d, sw128_kmajor_desc(a0 + k * 32), sw128_kmajor_desc(b0 + k * 32), idesc,
                            (kb | k) != 0 ? 1u : 0u);
          mma_commit_pair(&empty_c[s], 3);
        }
        mma_commit_pair(&acc_full[ab], 3);
      }
    }
  } else if (warp < kFirstEpiWarp) {
    // ------------------------------------------------------------ unpack warps
    const int cw = warp - kFirstConvWarp;
    const int grp = cw / kGroupWarps;
    const int tc = threadIdx.x - (kFirstConvWarp + grp * kGroupWarps) * 32;
    constexpr int NA = BM * 4 / kGroupThreads, NB = HB * 4 / kGroupThreads;
    const int rbase = tc >> 2, chunk = tc & 3;
    const uint32_t full_c_leader = mapa_shared(smem_u32(full_c), 0);
    int gbase = 0, it = 0;
    bool ok = true;
    for (int t = cluster_id_x(); t < p.tiles && ok; t += nclusters_x(), ++it, gbase += KB) {
      const int kb0 = ((grp - gbase) % kGroups + kGroups) % kGroups;
      uint32_t accA[NA], accB[NB];
#pragma unroll
      for (int j = 0; j < NA; ++j) accA[j] = 0;
#pragma unroll
      for (int j = 0; j < NB; ++j) accB[j] = 0;
      for (int kb = kb0; kb < KB; kb += kGroups) {
        const int g = gbase + kb;
        const int ps = g % P, c = g % SC;
        // the packed k-block (TMA, this CTA's 128 A rows then 128 B rows of 64 bytes)
        if (!PAIR_WAIT_CONV(&pack_full[ps], (g / P) & 1, abort_flag, &g_gemm_err)) {
          ok = false;
          break;
        }
        const uint8_t* pk = pack + ps * PACK_STAGE + rbase * BKP + chunk * 16;
        uint4 v[NA + NB];
#pragma unroll
        for (int j = 0; j < NA; ++j) v[j] = *reinterpret_cast<const uint4*>(pk + j * kRowStep * BKP);
#pragma unroll
        for (int j = 0; j < NB; ++j) v[NA + j] = *reinterpret_cast<const uint4*>(pk + A_PACK + j * kRowStep * BKP);
        __syncwarp();
        if (lane == 0) mbar_arrive(&pack_empty[ps]);
        // unpack into registers first: after the stage frees up only the stores remain
        Unpacked u[NA + NB];
#pragma unroll
        for (int j = 0; j < NA; ++j) u[j] = unpack_chunk(v[j], accA[j]);
#pragma unroll
        for (int j = 0; j < NB; ++j) u[NA + j] = unpack_chunk(v[NA + j], accB[j]);
        if (!PAIR_WAIT_CONV(&empty_c[c], ((g / SC) & 1) ^ 1, abort_flag, &g_gemm_err)) {
          ok = false;
          break;
        }
        uint8_t* ca = smem + c * CONV_STAGE;
        uint8_t* cb = ca + A_CONV;
#pragma unroll
        for (int j = 0; j < NA; ++j) store_chunk(u[j], ca, rbase + kRowStep * j, chunk);
#pragma unroll
        for (int j = 0; j < NB; ++j) store_chunk(u[NA + j], cb, rbase + kRowStep * j, chunk);
        fence_proxy_async_smem();
        __syncwarp();
        if (lane == 0) mbar_arrive_remote(full_c_leader + 8u * c);  // the leader's full_c[c]
      }
      if (!ok) break;
      // Row sums of u: A rows locally, B rows into this CTA's half of sumB in both CTAs.
      const int ab = it & 1;
      if (!mbar_wait_warp(&sums_empty[ab], ((it >> 1) & 1) ^ 1, abort_flag, &g_gemm_err)) break;
#pragma unroll
      for (int j = 0; j < NA; ++j) {
        int v = static_cast<int>(accA[j]);
        v += __shfl_xor_sync(0xFFFFFFFFu, v, 1);
        v += __shfl_xor_sync(0xFFFFFFFFu, v, 2);
        if (chunk == 0) sumA[(ab * kGroups + grp) * BM + rbase + kRowStep * j] = v;
      }
#pragma unroll
      for (int j = 0; j < NB; ++j) {
        int v = static_cast<int>(accB[j]);
        v += __shfl_xor_sync(0xFFFFFFFFu, v, 1);
        v += __shfl_xor_sync(0xFFFFFFFFu, v, 2);
        if (chunk == 0) {
          int* dst = &sumB[(ab * kGroups + grp) * BN + static_cast<int>(rank) * HB + rbase + kRowStep * j];
          *dst = v;
          st_shared_cluster_u32(mapa_shared(smem_u32(dst), peer), static_cast<uint32_t>(v));
        }
      }
      __syncwarp();
      if (lane == 0) {
        mbar_arrive_remote(mapa_shared(smem_u32(&sums_full[ab]), rank));
        mbar_arrive_remote(mapa_shared(smem_u32(&sums_full[ab]), peer));
      }
    }
  } else if (warp == kProducerWarp) {
    // ------------------------------------------------------------ producer: packed operands by TMA
    if (lane == 0) {
      tma_prefetch_desc(&tmA);
      tma_prefetch_desc(&tmB);
      int g = 0;
      bool ok = true;
      for (int t = cluster_id_x(); t < p.tiles && ok; t += nclusters_x()) {
        const int bz = t / per, r = t - bz * per, nb = r / p.num_m;
        const int m0 = (r - nb * p.num_m) * (2 * BM) + static_cast<int>(rank) * BM;  // this CTA's A rows
        const int n0 = nb * BN + static_cast<int>(rank) * HB;                       // this CTA's B rows
        for (int kb = 0; kb < min(KB, kPrefetchAhead); ++kb) {
          tma_prefetch_l2_3d(&tmA, kb * BKP, m0, bz);
          tma_prefetch_l2_3d(&tmB, kb * BKP, n0, bz);
        }
        for (int kb = 0; kb < KB; ++kb, ++g) {
          if (kb + kPrefetchAhead < KB) {
            tma_prefetch_l2_3d(&tmA, (kb + kPrefetchAhead) * BKP, m0, bz);
            tma_prefetch_l2_3d(&tmB, (kb + kPrefetchAhead) * BKP, n0, bz);
          }
          const int ps = g % P;
          if (!mbar_wait(&pack_empty[ps], ((g / P) & 1) ^ 1, abort_flag, &g_gemm_err)) {
            ok = false;
            break;
          }
          mbar_arrive_expect_tx(&pack_full[ps], PACK_STAGE);
          tma_load_3d(&tmA, &pack_full[ps], pack + ps * PACK_STAGE, kb * BKP, m0, bz);
          tma_load_3d(&tmB, &pack_full[ps], pack + ps * PACK_STAGE + A_PACK, kb * BKP, n0, bz);
        }
      }
      if (!ok) {
        // leave no TMA load in flight into this CTA's shared memory
        int fresh = 0;
        for (int j = (g > P ? g - P : 0); j < g; ++j)
          mbar_wait(&pack_full[j % P], (j / P) & 1, reinterpret_cast<volatile int*>(&fresh), &g_gemm_err,
                    100000000ull);
      }
    }
  } else {
    // ------------------------------------------------------------ epilogue warps
    const int ew = warp - kFirstEpiWarp;
    const int q = warp & 3;
    uint8_t* boxes = smem + OFF_STAGE + ew * 2 * BOX_BYTES;
    const uint32_t acc_empty_leader = mapa_shared(smem_u32(acc_empty), 0);
    int it = 0, nbox = 0;
    bool failed = false;
    for (int t = cluster_id_x(); t < p.tiles; t += nclusters_x(), ++it) {
      const int bz = t / per, r = t - bz * per, nb = r / p.num_m;
      const int m0 = (r - nb * p.num_m) * (2 * BM) + static_cast<int>(rank) * BM;
      const int n0 = nb * BN;
      const int ab = it & 1;
      const uint32_t ph = (it >> 1) & 1;
      if (!failed && !(mbar_wait_warp(&acc_full[ab], ph, abort_flag, &g_gemm_err) &&
                       mbar_wait_warp(&sums_full[ab], ph, abort_flag, &g_gemm_err)))
        failed = true;
      tc_fence_after();
      const int row = q * 32 + lane;
      const int m = m0 + row;
      epi_sync();
      if (!failed) {
        for (int i = ew * 32 + lane; i < BN; i += kEpiWarps * 32) {
          int v = 0;
#pragma unroll
          for (int q2 = 0; q2 < kGroups; ++q2) v += sumB[(ab * kGroups + q2) * BN + i];
          sbw[i] = static_cast<float>(-8 * v);
          if (MODE == static_cast<int>(GemmOut::kHalf)) colv[i] = (n0 + i < p.N) ? p.s_b[n0 + i] : 0.0f;
        }
      }
      epi_sync();
      if (failed) continue;
      int sa_u = 0;
#pragma unroll
      for (int q2 = 0; q2 < kGroups; ++q2) sa_u += sumA[(ab * kGroups + q2) * BM + row];
      const float corrA = static_cast<float>(64 * p.K - 8 * sa_u);
      const float sa = (MODE == static_cast<int>(GemmOut::kHalf) && m < p.M) ? p.s_a[m] : 0.0f;
#pragma unroll 1
      for (int cc = 0; cc < BN / 32; ++cc) {
        uint8_t* box = boxes + (nbox & 1) * BOX_BYTES;
        if (lane == 0) bulk_wait_group_read<1>();
        __syncwarp();
        uint8_t* rowp = box + lane * (32 * L::ELEM);
#pragma unroll 1
        for (int h = 0; h < 2; ++h) {
          const int c0 = cc * 32 + h * 16;
          uint32_t v[16];
          tmem_ld_32x32b_x16(tmem_base + (static_cast<uint32_t>(q * 32) << 16) + ab * BN + c0, v);
          tmem_ld_wait();
          if (cc == BN / 32 - 1 && h == 1) {
            tc_fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive_remote(acc_empty_leader + 8u * ab);
          }
          if (MODE == static_cast<int>(GemmOut::kHalf)) {
#pragma unroll
            for (int g2 = 0; g2 < 2; ++g2) {
              uint32_t w[4];
#pragma unroll
              for (int e = 0; e < 4; ++e) {
                const int i0 = g2 * 8 + 2 * e;
                const float a0 = __fmaf_rn(__uint_as_float(v[i0]), 262144.0f, corrA + sbw[c0 + i0]);
                const float a1 = __fmaf_rn(__uint_as_float(v[i0 + 1]), 262144.0f, corrA + sbw[c0 + i0 + 1]);
                const float y0 = __fmul_rn(__fmul_rn(a0, sa), colv[c0 + i0]);
                const float y1 = __fmul_rn(__fmul_rn(a1, sa), colv[c0 + i0 + 1]);
                const __half2 hh = __floats2half2_rn(y0, y1);
                w[e] = *reinterpret_cast<const uint32_t*>(&hh);
              }
              // 64-byte rows, 64-byte swizzle: 16-byte chunk (2h + g2) of row `lane`
              const int ch = 2 * h + g2;
              *reinterpret_cast<uint4*>(rowp + ((ch ^ ((lane >> 1) & 3)) << 4)) = make_uint4(w[0], w[1], w[2], w[3]);
            }
          } else {
#pragma unroll
            for (int g4 = 0; g4 < 4; ++g4) {
              uint32_t w[4];
#pragma unroll
              for (int e = 0; e < 4; ++e) {
                const int i = g4 * 4 + e;
                w[e] = static_cast<uint32_t>(
                    __float2int_rn(__fmaf_rn(__uint_as_float(v[i]), 262144.0f, corrA + sbw[c0 + i])));
              }
              // 128-byte rows, 128-byte swizzle: 16-byte chunk (4h + g4) of row `lane`
              const int ch = 4 * h + g4;
              *reinterpret_cast<uint4*>(rowp + ((ch ^ (lane & 7)) << 4)) = make_uint4(w[0], w[1], w[2], w[3]);
            }
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
      if (lane == 0) {
        mbar_arrive_remote(mapa_shared(smem_u32(&sums_empty[ab]), rank));
        mbar_arrive_remote(mapa_shared(smem_u32(&sums_empty[ab]), peer));
      }
    }
    if (lane == 0) bulk_wait_group_all();
    __syncwarp();
  }

  // Teardown: the pair's MMAs (which write both CTAs' TMEM) must be complete
  // before either CTA releases its TMEM.
  if (warp == 0 && lane == 0 && rank == 0 && *abort_flag) {
    for (int i = 0; i < 2; ++i) {
      const unsigned long long t0 = globaltimer();
      const uint32_t a = smem_u32(&acc_full[i]);
      while (!mbar_try_wait(a, 0) && !mbar_try_wait(a, 1) && globaltimer() - t0 < 100000000ull) {
      }
    }
  }
  tc_fence_before();
  cluster_sync();
  if (warp == 0) {
    tc_fence_after();
    tmem_dealloc_pair(tmem_base, TMEM_COLS);
  }
}

}  // namespace pair

}  // namespace

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

namespace {

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
  p.A = g.A;
  p.B = g.B;
  p.a_bs = g.a_batch_stride > 0 ? g.a_batch_stride : g.M;
  p.b_bs = g.b_batch_stride > 0 ? g.b_batch_stride : g.N;
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
  return launch_pdl(w4a4_gemm_kernel<BN, MODE>, dim3(grid), dim3(kThreads), C::SMEM, stream, ma, mb, md, p);
}

template <int MODE>
cudaError_t launch_pair(const GemmArgs& g, cudaStream_t stream) {
  static bool attr_set = false;
  if (!attr_set) {
    cudaError_t e = cudaFuncSetAttribute(pair::w4a4_gemm_pair_kernel<MODE>,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize, pair::Lay<MODE>::SMEM);
    if (e != cudaSuccess) return e;
    attr_set = true;
  }
  CUtensorMap ma, mb, md;
  if (!make_operand_map(&ma, g.A, g.K, g.M, g.batch, g.a_batch_stride, BM)) return cudaErrorInvalidValue;
  if (!make_operand_map(&mb, g.B, g.K, g.N, g.batch, g.b_batch_stride, pair::HB)) return cudaErrorInvalidValue;
  const int pitch = g.d_pitch > 0 ? g.d_pitch : g.N;
  if (!make_output_map(&md, g.D, g.out, g.M, g.N, pitch, g.batch)) return cudaErrorInvalidValue;
  Params p;
  p.A = g.A;
  p.B = g.B;
  p.a_bs = g.a_batch_stride > 0 ? g.a_batch_stride : g.M;
  p.b_bs = g.b_batch_stride > 0 ? g.b_batch_stride : g.N;
  p.M = g.M;
  p.N = g.N;
  p.K = g.K;
  p.batch = g.batch;
  p.num_m = (g.M + 2 * BM - 1) / (2 * BM);
  p.num_n = (g.N + pair::BN - 1) / pair::BN;
  p.tiles = p.num_m * p.num_n * g.batch;
  p.s_a = g.s_a;
  p.s_b = g.s_b;
  p.norm_a = g.norm_a;
  p.norm_b = g.norm_b;
  const int pairs = p.tiles < num_sms() / 2 ? p.tiles : num_sms() / 2;
  return launch_pdl(pair::w4a4_gemm_pair_kernel<MODE>, dim3(2 * pairs), dim3(pair::kPairThreads),
                    pair::Lay<MODE>::SMEM, stream, ma, mb, md, p);
}

}  // namespace

// CTA-pair kernel selection (a test hook; the default uses it for large fp16 linears).
static int g_pair_mode = -1;  // -1: automatic, 0: never, 1: whenever the shape allows

void set_gemm_pair_mode(int mode) { g_pair_mode = mode; }

cudaError_t launch_w4a4_gemm(const GemmArgs& g, cudaStream_t stream) {
  // a few rows (decode): weight streaming on the CUDA cores (automatic mode only)
  if (g_pair_mode == -1 && gemv_applies(g)) return launch_gemv(g, stream);
  const bool pair_ok = g.M > 0 && g.N >= 256 && g.batch > 0 && g_pair_mode != 0 &&
                       (g_pair_mode == 1 || (g.M >= 256 && g.out == GemmOut::kHalf));
  if (pair_ok && g.out == GemmOut::kHalf) return launch_pair<0>(g, stream);
  if (pair_ok && g.out == GemmOut::kS32) return launch_pair<1>(g, stream);
  // exact dot products of large token sets (the selector's Gram matrices):
  // the pair kernel as soon as both sides span a 256-row tile
  if (g_pair_mode != 0 && g.out == GemmOut::kS32 && g.M >= 256 && g.N >= 256 && g.batch > 0)
    return launch_pair<1>(g, stream);
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

namespace {

// One warp waits on an mbarrier that nothing ever arrives on. The bounded
// wait gives up after limit_ns and records kErrTimeout in the same device
// error word as the GEMM's waits, so the host sees exactly what a stalled
// GEMM pipeline would report; the kernel then returns normally.
__global__ void __launch_bounds__(32) expired_wait_kernel(unsigned long long limit_ns) {
  __shared__ __align__(8) uint64_t bar;
  __shared__ int abort_flag;
  if (threadIdx.x == 0) {
    mbar_init(&bar, 1);
    abort_flag = 0;
  }
  __syncthreads();
  mbar_wait_warp(&bar, 0, reinterpret_cast<volatile int*>(&abort_flag), &g_gemm_err, limit_ns);
}

}  // namespace

cudaError_t launch_expired_wait(unsigned long long limit_ns, cudaStream_t stream) {
  expired_wait_kernel<<<1, 32, 0, stream>>>(limit_ns);
  return cudaGetLastError();
}

unsigned int gemm_read_and_clear_error() {
  unsigned int v = 0, z = 0;
  cudaMemcpyFromSymbol(&v, g_gemm_err, sizeof(v));
  cudaMemcpyToSymbol(g_gemm_err, &z, sizeof(z));
  return v;
}

}  // namespace p4q
