// W4A4 integer GEMM on expanded operands (tcgen05 + TMEM + TMA, CTA pairs).
//
// Computes the same exact integer products and epilogues as p4q_gemm.cu
// (acc = P - 8 sum u_a - 8 sum u_b + 64 K from the FP8 product P of the
// offset codes u = v + 8), for linears large enough to be tensor-bound.
// Unpacking the nibbles inside the GEMM shares each SM's shared-memory path
// and issue slots with the MMAs and halves the rate the tensor pipe gets;
// here two streaming kernels first expand both packed operands into a
// caller workspace, one byte per code (the E4M3 byte u, exact), with the
// per-row sums of u, and the GEMM's operands then reach shared memory by TMA
// alone, already in the 128-byte-swizzled K-major layout the MMAs read.
//
// Byte order inside each 16-byte packed chunk (32 codes): for each packed
// 32-bit word, its four low-nibble codes, then its four high-nibble codes
// (p4q_expand.cu). The permutation is the same for both operands, so every
// dot product is unchanged.
//
// Operands [batch][rows][K] (row-contiguous, batch entries back to back),
// row sums [batch][rows], output [batch][M][pitch].
//
// int32 tiles may be narrower than 256 columns (p.bn, a multiple of 32): the
// selector's products of every token with its few kept tokens.
//
// Cosine-max tiles (MODE 2, the selector's initial diversity maxima of
// Eq. 4): the epilogue turns each row's exact dot products into its largest
// code cosine over the tile's columns and writes that one float per row and
// column tile (p.num_n partial maxima per row, p.part apart).
//
// Kernel: persistent, one cluster of two CTAs per 256 x 256 output tile,
//   warp 0    MMA issuer (leader CTA): 4 x tcgen05.mma (M 256, N 256, K 32)
//             per 128-deep k-block into one of two TMEM accumulators;
//   warp 1    producer: TMA of this CTA's 128 A rows and 128 B rows of a
//             k-block into a ring of stages; both CTAs' loads complete on the
//             leader's barrier (cta_group::2 form of the TMA load);
//   warps 2-5 epilogue, overlapped with the next tile: TMEM loads, the exact
//             correction from the row sums, scales, fp16 or int32 boxes
//             stored by TMA.
#include <cuda.h>
#include <cudaTypedefs.h>
#include <cuda_fp16.h>

#include <algorithm>

#include "p4q_device.cuh"
#include "p4q_internal.h"

namespace p4q {

__device__ unsigned int g_gemm8_err;

namespace {

constexpr int BM = 128;                 // A rows per CTA (TMEM lanes)
constexpr int BN = 256;                 // output columns per pair tile
constexpr int HB = BN / 2;              // B rows per CTA
constexpr int BK = 128;                 // k (bytes of expanded codes) per stage
constexpr int A_BYTES = BM * BK;
constexpr int STAGE_BYTES = (BM + HB) * BK;
constexpr int kEpiWarps = 4;
constexpr int kFirstEpiWarp = 2;
constexpr int kThreads = (kFirstEpiWarp + kEpiWarps) * 32;
constexpr uint32_t TMEM_COLS = 2 * BN;
constexpr int kMinRows = 512;           // smaller M: the in-kernel unpack path is cheaper than the expansion

struct Params8 {
  int M, N, K, batch;
  int num_m, num_n, per, tiles;  // per: tiles per batch entry
  int bn;                        // int32 tiles: output columns per pair tile (<= BN)
  int gm;                        // row tiles per raster group (tile_coords)
  int f32_out;                   // int32 tiles: store the exact integers as fp32 values instead
  const float* s_a;
  const float* s_b;
  const int32_t* sum_a;  // [batch, M] sum of u over each A row
  const int32_t* sum_b;  // [batch, N]
  const int32_t* norm_a;  // cosine-max tiles: [batch, M] squared code norms of the A rows
  const int32_t* norm_b;  // [batch, N] of the B rows
  float* cos_max;         // [num_n][part] with part >= batch * M: each A row's largest cosine per column tile
  size_t part;
  uint32_t* rowmax;       // fp16 tiles: [rm_n, M] each row's largest |Y| bit pattern per column range
  int rm_n;
  int rm_c0[2], rm_c1[2];
};

constexpr int kCosMode = static_cast<int>(GemmOut::kCos);

template <int MODE>  // GemmOut::kHalf, kS32 or kCos
struct Lay8 {
  static constexpr int ELEM = (MODE == static_cast<int>(GemmOut::kHalf)) ? 2 : 4;
  static constexpr int BOX_BYTES = 32 * 32 * ELEM;
  static constexpr int FIXED = kEpiWarps * 2 * BOX_BYTES + 2 * BN * 4 + 512;
  static constexpr int S_FIT = (232448 - 1024 - FIXED) / STAGE_BYTES;
  static constexpr int S = S_FIT > 8 ? 8 : S_FIT;
  static constexpr int OFF_BOX = S * STAGE_BYTES;
  static constexpr int OFF_COL = OFF_BOX + kEpiWarps * 2 * BOX_BYTES;  // colv[BN], sbw[BN]
  static constexpr int OFF_BAR = OFF_COL + 2 * BN * 4;
  static constexpr int NBAR = 2 * S + 4;
  static constexpr int OFF_MISC = OFF_BAR + NBAR * 8;
  static constexpr int SMEM = 1024 + OFF_MISC + 16;
  static_assert(S >= 3, "TMA stages");
  static_assert(SMEM <= 232448, "shared memory budget");
};

// Tile t -> (batch entry, row tile, column tile). Narrow int32 tiles (bn <
// BN: a few column tiles over a short B) vary their column tile fastest, so
// that the pairs reading the same A rows run side by side. Otherwise the row
// tiles are rastered in groups of p.gm: consecutive tiles sweep a group's row
// tiles, then the next column tile, so a group's A rows (sized to stay in L2)
// are read from DRAM once while the group sweeps all of B; p.gm = 1 (a B
// that fits L2) is plain row-major order.
__device__ __forceinline__ void tile_coords(const Params8& p, int t, int* bz, int* mt, int* nb) {
  *bz = t / p.per;
  const int r = t - *bz * p.per;
  if (p.bn < BN) {
    *mt = r / p.num_n;
    *nb = r - *mt * p.num_n;
  } else {
    const int span = p.gm * p.num_n;  // tiles of a full group
    const int grp = r / span;
    const int gm = min(p.gm, p.num_m - grp * p.gm);
    const int q = r - grp * span;
    *nb = q / gm;
    *mt = grp * p.gm + (q - *nb * gm);
  }
}

__device__ __forceinline__ void epi_sync8() {
  asm volatile("bar.sync 1, %0;" ::"n"(kEpiWarps * 32) : "memory");
}

// 3-D TMA load into this CTA's shared memory whose completion is counted on
// an mbarrier of either CTA of the pair (cta_group::2 form).
__device__ __forceinline__ void tma_load_3d_pair(const CUtensorMap* map, uint32_t bar_cluster, void* smem_dst, int c0,
                                                 int c1, int c2) {
  asm volatile(
      "cp.async.bulk.tensor.3d.cta_group::2.shared::cluster.global.tile.mbarrier::complete_tx::bytes"
      " [%0], [%1, {%3, %4, %5}], [%2];" ::"r"(smem_u32(smem_dst)),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(bar_cluster), "r"(c0), "r"(c1), "r"(c2)
      : "memory");
}

template <int MODE>
__global__ void __cluster_dims__(2, 1, 1) __launch_bounds__(kThreads, 1)
    w4a4_gemm8_pair_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB,
                           const __grid_constant__ CUtensorMap tmD, const Params8 p) {
  using L = Lay8<MODE>;
  constexpr int S = L::S, BOX_BYTES = L::BOX_BYTES;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + L::OFF_BAR);
  uint64_t* full = bars;               // [S] leader: both CTAs' TMA bytes of a stage
  uint64_t* empty = full + S;          // [S] MMA commit (both CTAs) -> producers
  uint64_t* acc_full = empty + S;      // [2] MMA commit (both CTAs) -> epilogues
  uint64_t* acc_empty = acc_full + 2;  // [2] leader: both CTAs' epilogues -> MMA
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(smem + L::OFF_MISC);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(smem + L::OFF_MISC + 4);
  float* colv = reinterpret_cast<float*>(smem + L::OFF_COL);
  float* sbw = colv + BN;

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const uint32_t rank = cluster_ctarank();
  const int KB = p.K / BK;
  const int bn = (MODE != static_cast<int>(GemmOut::kHalf)) ? p.bn : BN;  // columns of a pair tile
  const int hb = bn / 2;                                                  // B rows per CTA

  if (threadIdx.x == 0) {
    for (int i = 0; i < S; ++i) {
      mbar_init(&full[i], 1);  // the leader's expect_tx arrival; both CTAs' bytes
      mbar_init(&empty[i], 1);
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(&acc_full[i], 1);
      mbar_init(&acc_empty[i], 2 * kEpiWarps);
    }
    *abort_flag = 0;
    fence_barrier_init();
  }
  if (warp == 0) {
    tmem_alloc_pair(tmem_slot, TMEM_COLS);
    tmem_relinquish_pair();
  }
  tc_fence_before();
  cluster_sync();
  tc_fence_after();
  const uint32_t tmem_base = *tmem_slot;
  pdl_wait();  // expanded operands and scales come from the previous kernels
  pdl_launch_dependents();

  if (warp == 0) {
    // ------------------------------------------------------------ MMA issuer (leader)
    if (lane == 0 && rank == 0) {
      const uint32_t idesc = idesc_e4m3_f32(2 * BM, bn);
      int g = 0, it = 0;
      bool ok = true;
      for (int t = cluster_id_x(); t < p.tiles && ok; t += nclusters_x(), ++it) {
        const int ab = it & 1;
        if (!mbar_wait(&acc_empty[ab], ((it >> 1) & 1) ^ 1, abort_flag, &g_gemm8_err)) break;
        tc_fence_after();
        const uint32_t d = tmem_base + static_cast<uint32_t>(ab * BN);
        for (int kb = 0; kb < KB; ++kb, ++g) {
          const int s = g % S;
          if (!mbar_wait_spin(&full[s], (g / S) & 1, abort_flag, &g_gemm8_err)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t a0 = smem_u32(smem + s * STAGE_BYTES);
          const uint32_t b0 = a0 + A_BYTES;
#pragma unroll
          for (int k = 0; k < BK / 32; ++k)
            mma_f8f6f4_pair(d, sw128_kmajor_desc(a0 + k * 32), sw128_kmajor_desc(b0 + k * 32), idesc,
                            (kb | k) != 0 ? 1u : 0u);
          mma_commit_pair(&empty[s], 3);
        }
        if (!ok) break;
        mma_commit_pair(&acc_full[ab], 3);
      }
    }
  } else if (warp == 1) {
    // ------------------------------------------------------------ producer
    if (lane == 0) {
      tma_prefetch_desc(&tmA);
      tma_prefetch_desc(&tmB);
      const uint32_t full_leader = mapa_shared(smem_u32(full), 0);
      int g = 0;
      bool ok = true;
      for (int t = cluster_id_x(); t < p.tiles && ok; t += nclusters_x()) {
        int bz, mt, nb;
        tile_coords(p, t, &bz, &mt, &nb);
        const int m0 = mt * (2 * BM) + static_cast<int>(rank) * BM;  // this CTA's A rows
        const int n0 = nb * bn + static_cast<int>(rank) * hb;                       // this CTA's B rows
        for (int kb = 0; kb < KB; ++kb, ++g) {
          const int s = g % S;
          if (!mbar_wait_spin(&empty[s], ((g / S) & 1) ^ 1, abort_flag, &g_gemm8_err)) {
            ok = false;
            break;
          }
          if (rank == 0) mbar_arrive_expect_tx(&full[s], 2 * (A_BYTES + hb * BK));
          uint8_t* st = smem + s * STAGE_BYTES;
          tma_load_3d_pair(&tmA, full_leader + 8u * s, st, kb * BK, m0, bz);
          tma_load_3d_pair(&tmB, full_leader + 8u * s, st + A_BYTES, kb * BK, n0, bz);
        }
      }
      if (!ok && rank == 0) {
        // leave no TMA load in flight into the pair's shared memory
        int fresh = 0;
        for (int j = (g > S ? g - S : 0); j < g; ++j)
          mbar_wait(&full[j % S], (j / S) & 1, reinterpret_cast<volatile int*>(&fresh), &g_gemm8_err,
                    100000000ull);
      }
    }
  } else if (MODE == kCosMode) {
    // ------------------------------------------------------------ epilogue warps: cosine max per row
    const int ew = warp - kFirstEpiWarp;
    const int q = warp & 3;  // TMEM lane quarter of this warp
    int32_t* cnr = reinterpret_cast<int32_t*>(smem + L::OFF_BOX);  // [BN] B norms
    float* cbias = reinterpret_cast<float*>(cnr + BN);              // [BN] 0, or -inf past N
    const uint32_t acc_empty_leader = mapa_shared(smem_u32(acc_empty), 0);
    int it = 0;
    bool failed = false;
    for (int t = cluster_id_x(); t < p.tiles; t += nclusters_x(), ++it) {
      int bz, mt, nb;
      tile_coords(p, t, &bz, &mt, &nb);
      const int m0 = mt * (2 * BM) + static_cast<int>(rank) * BM;
      const int n0 = nb * bn;
      const int ab = it & 1;
      if (!failed && !mbar_wait_warp(&acc_full[ab], (it >> 1) & 1, abort_flag, &g_gemm8_err)) failed = true;
      tc_fence_after();
      epi_sync8();  // every epilogue warp is done with the previous tile's column constants
      if (!failed) {
        for (int i = ew * 32 + lane; i < bn; i += kEpiWarps * 32) {
          const int n = n0 + i;
          const size_t nn = static_cast<size_t>(bz) * p.N + n;
          const bool in = n < p.N;
          const int nbv = in ? p.norm_b[nn] : 0;
          sbw[i] = in ? static_cast<float>(-8 * p.sum_b[nn]) : 0.0f;
          cnr[i] = nbv;
          colv[i] = nbv > 0 ? rsqrtf(static_cast<float>(nbv)) : 0.0f;
          cbias[i] = in ? 0.0f : -INFINITY;  // zero-filled B rows past N take no part
        }
      }
      epi_sync8();
      if (failed) continue;
      const int m = m0 + q * 32 + lane;
      const bool row_in = m < p.M;
      const size_t ma = static_cast<size_t>(bz) * p.M + m;
      const float corrA = row_in ? static_cast<float>(64 * p.K - 8 * p.sum_a[ma]) : 0.0f;
      const int na = row_in ? p.norm_a[ma] : 0;
      const float ra = na > 0 ? rsqrtf(static_cast<float>(na)) : 0.0f;
      const uint32_t taddr = tmem_base + (static_cast<uint32_t>(q * 32) << 16) + ab * BN;
      // Pass 1: the largest approximate cosine (as dot * rsqrt(na) * rsqrt(nb),
      // within cos_approx's error bound), the runner-up, and the dot product at
      // the largest. Only columns within kCosMargin of the largest can hold the
      // exact maximum; when the runner-up is not among them, the exact maximum
      // is the largest column's code cosine.
      float amax = -INFINITY, a2 = -INFINITY, xarg = 0.0f;
      int carg = 0;
#pragma unroll 1
      for (int c0 = 0; c0 < bn; c0 += 32) {
        uint32_t v[32];
        tmem_ld_32x32b_x32(taddr + c0, v);
        tmem_ld_wait();
#pragma unroll
        for (int i = 0; i < 32; ++i) {
          const int c = c0 + i;
          const float x = __fmaf_rn(__uint_as_float(v[i]), 262144.0f, corrA + sbw[c]);  // exact dot
          const float ap = __fmul_rn(__fmul_rn(x, ra), colv[c]) + cbias[c];
          a2 = fmaxf(a2, fminf(ap, amax));
          if (ap > amax) {
            amax = ap;
            xarg = x;
            carg = c;
          }
        }
      }
      const bool slow = a2 >= amax - kCosMargin;
      float emax = code_cosine(static_cast<int>(xarg), na, cnr[carg]);
      if (__any_sync(0xFFFFFFFFu, slow)) {
        // Pass 2 (near ties): the exact cosine of every column within the margin
        float e2 = -INFINITY;
#pragma unroll 1
        for (int c0 = 0; c0 < bn; c0 += 32) {
          uint32_t v[32];
          tmem_ld_32x32b_x32(taddr + c0, v);
          tmem_ld_wait();
          if (slow) {
#pragma unroll
            for (int i = 0; i < 32; ++i) {
              const int c = c0 + i;
              const float x = __fmaf_rn(__uint_as_float(v[i]), 262144.0f, corrA + sbw[c]);
              const float ap = __fmul_rn(__fmul_rn(x, ra), colv[c]) + cbias[c];
              if (ap >= amax - kCosMargin) e2 = fmaxf(e2, code_cosine(static_cast<int>(x), na, cnr[c]));
            }
          }
        }
        if (slow) emax = e2;
      }
      // the accumulator is free for the next tile
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive_remote(acc_empty_leader + 8u * ab);
      if (row_in) p.cos_max[static_cast<size_t>(nb) * p.part + ma] = emax;
    }
  } else {
    // ------------------------------------------------------------ epilogue warps
    const int ew = warp - kFirstEpiWarp;
    const int q = warp & 3;  // TMEM lane quarter of this warp
    uint8_t* boxes = smem + L::OFF_BOX + ew * 2 * BOX_BYTES;
    const uint32_t acc_empty_leader = mapa_shared(smem_u32(acc_empty), 0);
    int it = 0, nbox = 0;
    bool failed = false;
    for (int t = cluster_id_x(); t < p.tiles; t += nclusters_x(), ++it) {
      int bz, mt, nb;
      tile_coords(p, t, &bz, &mt, &nb);
      const int m0 = mt * (2 * BM) + static_cast<int>(rank) * BM;
      const int n0 = nb * bn;
      const int ab = it & 1;
      if (!failed && !mbar_wait_warp(&acc_full[ab], (it >> 1) & 1, abort_flag, &g_gemm8_err)) failed = true;
      tc_fence_after();
      const int row = q * 32 + lane;
      const int m = m0 + row;
      epi_sync8();  // every epilogue warp is done with the previous tile's column constants
      if (!failed) {
        for (int i = ew * 32 + lane; i < bn; i += kEpiWarps * 32) {
          const int n = n0 + i;
          sbw[i] = (n < p.N) ? static_cast<float>(-8 * p.sum_b[static_cast<size_t>(bz) * p.N + n]) : 0.0f;
          if (MODE == static_cast<int>(GemmOut::kHalf)) colv[i] = (n < p.N) ? p.s_b[n] : 0.0f;
        }
      }
      epi_sync8();
      if (failed) continue;
      // acc = P - 8 sum u_a - 8 sum u_b + 64 K in fp32: every term and partial
      // result is an integer of magnitude < 2^24, so the fused multiply-add is exact.
      const float corrA = (m < p.M) ? static_cast<float>(64 * p.K - 8 * p.sum_a[static_cast<size_t>(bz) * p.M + m]) : 0.0f;
      const float sa = (MODE == static_cast<int>(GemmOut::kHalf) && m < p.M) ? p.s_a[m] : 0.0f;
      uint32_t rmx0 = 0, rmx1 = 0;  // fp16 tiles: |Y| bit-pattern maxima (two halfwords) per column range
#pragma unroll 1
      for (int cc = 0; cc < bn / 32; ++cc) {
        uint8_t* box = boxes + (nbox & 1) * BOX_BYTES;
        uint32_t cmx = 0;
        if (lane == 0) bulk_wait_group_read<1>();
        __syncwarp();
        uint8_t* rowp = box + lane * (32 * L::ELEM);
#pragma unroll 1
        for (int h = 0; h < 2; ++h) {
          const int c0 = cc * 32 + h * 16;
          uint32_t v[16];
          tmem_ld_32x32b_x16(tmem_base + (static_cast<uint32_t>(q * 32) << 16) + ab * BN + c0, v);
          tmem_ld_wait();
          if (cc == bn / 32 - 1 && h == 1) {
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
                cmx = __vmaxu2(cmx, w[e] & 0x7FFF7FFFu);
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
                const float x = __fmaf_rn(__uint_as_float(v[i]), 262144.0f, corrA + sbw[c0 + i]);
                w[e] = p.f32_out ? __float_as_uint(x) : static_cast<uint32_t>(__float2int_rn(x));
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
        if (MODE == static_cast<int>(GemmOut::kHalf) && p.rm_n > 0) {
          // this 32-column chunk lies wholly inside or outside each range (multiples of 32)
          const int c = n0 + cc * 32;
          if (c >= p.rm_c0[0] && c < p.rm_c1[0]) rmx0 = __vmaxu2(rmx0, cmx);
          if (p.rm_n > 1 && c >= p.rm_c0[1] && c < p.rm_c1[1]) rmx1 = __vmaxu2(rmx1, cmx);
        }
      }
      if (MODE == static_cast<int>(GemmOut::kHalf) && p.rm_n > 0 && m < p.M) {
        // one atomic per row and range the tile meets
        if (n0 < p.rm_c1[0] && n0 + bn > p.rm_c0[0])
          atomicMax(p.rowmax + m, max(rmx0 & 0xFFFFu, rmx0 >> 16));
        if (p.rm_n > 1 && n0 < p.rm_c1[1] && n0 + bn > p.rm_c0[1])
          atomicMax(p.rowmax + static_cast<size_t>(p.M) + m, max(rmx1 & 0xFFFFu, rmx1 >> 16));
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

// 3-D map over expanded codes: dims (K bytes, rows, batch), 128 x box_rows
// boxes, 128-byte swizzle (the K-major layout the MMA descriptors describe).
bool make_expanded_map(CUtensorMap* map, const uint8_t* base, int K, int rows, int batch, int box_rows) {
  auto enc = get_encode_fn();
  if (!enc) return false;
  cuuint64_t dims[3] = {static_cast<cuuint64_t>(K), static_cast<cuuint64_t>(rows), static_cast<cuuint64_t>(batch)};
  cuuint64_t strides[2] = {static_cast<cuuint64_t>(K), static_cast<cuuint64_t>(K) * rows};
  cuuint32_t box[3] = {static_cast<cuuint32_t>(BK), static_cast<cuuint32_t>(box_rows), 1};
  cuuint32_t estr[3] = {1, 1, 1};
  return enc(map, CU_TENSOR_MAP_DATA_TYPE_UINT8, 3, const_cast<uint8_t*>(base), dims, strides, box, estr,
             CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
             CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

size_t align256(size_t x) { return (x + 255) & ~static_cast<size_t>(255); }

struct Ws8 {
  uint8_t* a8;
  uint8_t* b8;
  int32_t* sum_a;
  int32_t* sum_b;
};

size_t ws8_layout(int M, int N, int K, void* base, Ws8* w) {
  const size_t oa = 0;
  const size_t ob = align256(oa + static_cast<size_t>(M) * K);
  const size_t osa = align256(ob + static_cast<size_t>(N) * K);
  const size_t osb = align256(osa + static_cast<size_t>(M) * 4);
  const size_t end = align256(osb + static_cast<size_t>(N) * 4);
  if (base && w) {
    uint8_t* b = static_cast<uint8_t*>(base);
    w->a8 = b + oa;
    w->b8 = b + ob;
    w->sum_a = reinterpret_cast<int32_t*>(b + osa);
    w->sum_b = reinterpret_cast<int32_t*>(b + osb);
  }
  return end;
}

template <int MODE>
cudaError_t launch8(const GemmArgs& g, const Ws8& w, cudaStream_t stream) {
  const int bn = (MODE != static_cast<int>(GemmOut::kHalf)) ? g.tile_n : BN;
  if (bn < 32 || bn > BN || bn % 32 != 0) return cudaErrorInvalidValue;
  if (MODE == kCosMode && (!g.norm_a || !g.norm_b || !g.D)) return cudaErrorInvalidValue;
  static bool attr_set = false;
  if (!attr_set) {
    cudaError_t e = cudaFuncSetAttribute(w4a4_gemm8_pair_kernel<MODE>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         Lay8<MODE>::SMEM);
    if (e != cudaSuccess) return e;
    attr_set = true;
  }
  CUtensorMap ma, mb, md;
  const int batch = g.batch > 0 ? g.batch : 1;
  if (!make_expanded_map(&ma, w.a8, g.K, g.M, batch, BM)) return cudaErrorInvalidValue;
  if (!make_expanded_map(&mb, w.b8, g.K, g.N, batch, bn / 2)) return cudaErrorInvalidValue;
  if (MODE == kCosMode) {
    md = ma;  // no tiles are stored: one float per A row and column tile
  } else {
    const int pitch = g.d_pitch > 0 ? g.d_pitch : g.N;
    // a row narrower than 16 bytes is stored over its whole pitch (the extra
    // columns hold the products with zero-filled B rows)
    const int ocols = (g.N * 4 < 16) ? pitch : g.N;
    if (!make_output_map(&md, g.D, g.out, g.M, ocols, pitch, batch)) return cudaErrorInvalidValue;
  }
  Params8 p;
  p.M = g.M;
  p.N = g.N;
  p.K = g.K;
  p.batch = batch;
  p.num_m = (g.M + 2 * BM - 1) / (2 * BM);
  p.num_n = (g.N + bn - 1) / bn;
  p.bn = bn;
  // Raster: a B of at most 32 MB stays in L2 while the row tiles stream past
  // it (row-major order, every A row read once; measured: a 71 MB B did not
  // stay, as the L2 is split between the two dies); a larger B is swept by
  // groups of row tiles whose A rows (about 24 MB) stay in L2.
  const bool b_fits = static_cast<size_t>(g.N) * g.K <= (32u << 20);
  p.gm = b_fits ? 1
                : std::max(1, std::min(p.num_m, static_cast<int>((24u << 20) / (static_cast<size_t>(2 * BM) * g.K))));
  p.f32_out = g.f32_out ? 1 : 0;
  p.per = p.num_m * p.num_n;
  p.tiles = p.per * batch;
  p.s_a = g.s_a;
  p.s_b = g.s_b;
  p.sum_a = w.sum_a;
  p.sum_b = w.sum_b;
  p.norm_a = g.norm_a;
  p.norm_b = g.norm_b;
  p.cos_max = MODE == kCosMode ? static_cast<float*>(g.D) : nullptr;
  p.part = static_cast<size_t>(batch) * g.M;
  p.rowmax = g.rowmax;
  p.rm_n = (MODE == static_cast<int>(GemmOut::kHalf) && g.rowmax && batch == 1) ? g.rm_n : 0;
  for (int r = 0; r < 2; ++r) {
    p.rm_c0[r] = g.rm_c0[r];
    p.rm_c1[r] = g.rm_c1[r];
  }
  const int pairs = p.tiles < num_sms() / 2 ? p.tiles : num_sms() / 2;
  return launch_pdl(w4a4_gemm8_pair_kernel<MODE>, dim3(2 * pairs), dim3(kThreads), Lay8<MODE>::SMEM, stream, ma,
                    mb, md, p);
}

}  // namespace

size_t gemm8_workspace_bytes(int M, int N, int K) { return ws8_layout(M, N, K, nullptr, nullptr); }

static int g_gemm8_mode = 0;  // 0 automatic, 1 never, 2 whenever a workspace is given (tests)

void set_gemm8_mode(int mode) { g_gemm8_mode = mode; }

bool gemm8_applies(const GemmArgs& g) {
  if (g_gemm8_mode == 1) return false;
  if (g.batch != 1 || g.M <= 0 || g.N < 256 || (g.out != GemmOut::kHalf && g.out != GemmOut::kS32)) return false;
  return g_gemm8_mode == 2 || g.M >= kMinRows;
}

cudaError_t launch_gemm8(const GemmArgs& g, const uint8_t* a8, const int32_t* sum_a, const uint8_t* b8,
                         const int32_t* sum_b, cudaStream_t stream) {
  Ws8 w;
  w.a8 = const_cast<uint8_t*>(a8);
  w.b8 = const_cast<uint8_t*>(b8);
  w.sum_a = const_cast<int32_t*>(sum_a);
  w.sum_b = const_cast<int32_t*>(sum_b);
  switch (g.out) {
    case GemmOut::kHalf: return launch8<0>(g, w, stream);
    case GemmOut::kS32: return launch8<1>(g, w, stream);
    default: return launch8<kCosMode>(g, w, stream);
  }
}

cudaError_t launch_w4a4_gemm8(const GemmArgs& g, void* ws, size_t ws_bytes, cudaStream_t stream) {
  Ws8 w;
  if (!ws || ws_bytes < ws8_layout(g.M, g.N, g.K, ws, &w)) return cudaErrorInvalidValue;
  cudaError_t e = launch_expand_codes(g.A, g.M, g.K, w.a8, w.sum_a, stream);
  if (e != cudaSuccess) return e;
  e = launch_expand_codes(g.B, g.N, g.K, w.b8, w.sum_b, stream);
  if (e != cudaSuccess) return e;
  return launch_gemm8(g, w.a8, w.sum_a, w.b8, w.sum_b, stream);
}

unsigned int gemm8_read_and_clear_error() {
  unsigned int v = 0, z = 0;
  cudaMemcpyFromSymbol(&v, g_gemm8_err, sizeof(v));
  cudaMemcpyToSymbol(g_gemm8_err, &z, sizeof(z));
  return v;
}

}  // namespace p4q
