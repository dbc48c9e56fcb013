// Causal softmax attention on the pruned sequence with FP16 keys and values
// (App. B: the language model's linears run in W4A4 while the key and value
// caches stay in FP16). Per sample of m positions and per head h:
//   o_i = sum_{j <= i} p_ij v_j,  p_i. = softmax_j(q_i . k_j / sqrt(d_h)),
// key/value head h / (H / H_kv).
//
// One CTA per (128-query block, head, sample), 16 warps: warp w reads TMEM
// lanes 32 (w % 4) .. + 31 (query rows) and takes every fourth 32-column
// chunk from chunk w / 4 on (keys for S, head dimensions for O):
//   1. thread 0 loads the query block (128 x 128 fp16) and the keys 0 .. nk-1
//      the block can see (nk rounded up to 64) by TMA into 128-byte swizzled
//      K-major tiles, and issues S = Q K^T on the tensor cores (tcgen05,
//      kind::f16, fp32 accumulators in TMEM columns 0 .. nk-1);
//   2. the values of the same keys arrive by TMA too, one 16 KB block per 64
//      keys in the space of its V^T tile; once they are in, every thread
//      takes an 8 x 8 block of a tile into registers, and after a block-wide
//      barrier writes it back transposed, so that each tile becomes K-major
//      V^T (128 rows of head dimensions x 64 keys); keys at or past m are
//      zero;
//   3. each warp reads its chunks of S from TMEM twice: the row maxima of the
//      four warps sharing the rows meet in shared memory, then
//      p = 2^((s - max) log2(e) / sqrt(d_h)) (p = 0 past the causal limit) is
//      written as fp16 into K-major tiles in the space the keys used, and the
//      partial row sums meet in shared memory;
//   4. thread 0 issues O = P V (fp32 in TMEM columns 0 .. 127, which S no
//      longer needs); each warp scales its 32 columns by 1 / sum and stores
//      fp16.
// Every wait is bounded; a time-out sets the kernel's device error word.
#include <cuda_fp16.h>

#include "p4q.h"
#include "p4q_device.cuh"
#include "p4q_internal.h"

namespace p4q {

__device__ unsigned int g_attn_err;

namespace {

constexpr int kBQ = 128;        // query rows per CTA
constexpr int kDH = 128;        // head dimension
constexpr int kKeyBlock = 64;   // keys per P / V^T tile
constexpr int kThreads = 512;
constexpr int kLaneGroups = 4;     // warps w and w + 4k share TMEM lanes 32 (w % 4) ..
constexpr int kTileBytes = 16384;  // 128 rows x 128 bytes

struct AttnParams {
  __half* o;
  long long ldo;
  int m, group, nkmax;
  float c2;  // log2(e) / sqrt(d_h)
};

// Instruction descriptor of kind::f16 with fp16 A and B (both K-major) and an
// fp32 accumulator, for an M x N tile.
__host__ __device__ constexpr uint32_t idesc_f16_f32(int M, int N) {
  return (1u << 4)                                 // D format F32
         | (0u << 7) | (0u << 10)                  // A, B format F16
         | (static_cast<uint32_t>(N >> 3) << 17)   // N / 8
         | (static_cast<uint32_t>(M >> 4) << 24);  // M / 16
}

__device__ __forceinline__ void mma_f16(uint32_t d_tmem, uint64_t a_desc, uint64_t b_desc, uint32_t idesc,
                                        uint32_t accumulate) {
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "setp.ne.b32 p, %4, 0;\n\t"
      "tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n\t}\n" ::"r"(d_tmem),
      "l"(a_desc), "l"(b_desc), "r"(idesc), "r"(accumulate)
      : "memory");
}

// Byte offset of 16-byte chunk c of row r in a 128-byte swizzled K-major tile.
__device__ __forceinline__ uint32_t sw128_off(int r, int c) {
  return static_cast<uint32_t>((r >> 3) * 1024 + (r & 7) * 128 + ((c ^ (r & 7)) << 4));
}

__global__ void __launch_bounds__(kThreads, 1)
    causal_attention_kernel(const __grid_constant__ CUtensorMap tmQ, const __grid_constant__ CUtensorMap tmK,
                            const __grid_constant__ CUtensorMap tmV, const AttnParams p) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  const int nkmax = p.nkmax;
  uint8_t* sQ = smem;                                    // 2 tiles: head dims 0-63, 64-127
  uint8_t* sKP = smem + 2 * kTileBytes;                  // K: 2 x [nkmax x 128 B]; later P tiles
  uint8_t* sVt = sKP + static_cast<size_t>(nkmax) * 256;  // V^T tiles, one per 64 keys
  uint64_t* bars = reinterpret_cast<uint64_t*>(sVt + static_cast<size_t>(nkmax) * 256);
  uint64_t* tma_bar = bars;
  uint64_t* mma_bar = bars + 1;
  uint64_t* v_bar = bars + 2;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + 3);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(bars + 4);
  // [4][128] partial row maxima, then row sums: in the query tiles, which S = Q K^T no longer needs
  float* red = reinterpret_cast<float*>(sQ);

  const int qb = blockIdx.x, h = blockIdx.y, b = blockIdx.z;
  const int hk = h / p.group;
  const int t = threadIdx.x, warp = t >> 5;
  const int m = p.m;
  const int last_key = min(m, (qb + 1) * kBQ) - 1;            // the block's last visible key
  const int nk = ((last_key + kKeyBlock) / kKeyBlock) * kKeyBlock;  // keys loaded, multiple of 64
  const uint32_t tmem_cols = nkmax <= 128 ? 128u : nkmax <= 256 ? 256u : 512u;

  if (t == 0) {
    mbar_init(tma_bar, 1);
    mbar_init(mma_bar, 1);
    mbar_init(v_bar, 1);
    *abort_flag = 0;
    fence_barrier_init();
  }
  if (warp == 0) {
    tmem_alloc(tmem_slot, tmem_cols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  pdl_wait();
  pdl_launch_dependents();

  // ---------------------------------------------------------------- 1. loads and S = Q K^T
  if (t == 0) {
    tma_prefetch_desc(&tmQ);
    tma_prefetch_desc(&tmK);
    tma_prefetch_desc(&tmV);
    mbar_arrive_expect_tx(v_bar, static_cast<uint32_t>(nk * 256));
    // V block j (64 keys x 128 dims) -> tile j: dims 0-63 in its first 8 KB, 64-127 in the second
    for (int r0 = 0; r0 < nk; r0 += kKeyBlock)
      for (int kb = 0; kb < 2; ++kb)
        tma_load_3d(&tmV, v_bar, sVt + (r0 / kKeyBlock) * kTileBytes + kb * 8192, hk * kDH + kb * 64, b * m + r0, 0);
    mbar_arrive_expect_tx(tma_bar, static_cast<uint32_t>(2 * kTileBytes + nk * 256));
    const int row_q = b * m + qb * kBQ, row_k = b * m;
#pragma unroll
    for (int kb = 0; kb < 2; ++kb) tma_load_3d(&tmQ, tma_bar, sQ + kb * kTileBytes, h * kDH + kb * 64, row_q, 0);
    for (int kb = 0; kb < 2; ++kb)
      for (int r0 = 0; r0 < nk; r0 += kKeyBlock)
        tma_load_3d(&tmK, tma_bar, sKP + static_cast<size_t>(kb) * nkmax * 128 + r0 * 128, hk * kDH + kb * 64,
                    row_k + r0, 0);
    if (mbar_wait(tma_bar, 0, abort_flag, &g_attn_err)) {
      tc_fence_after();
      constexpr uint32_t idesc = idesc_f16_f32(kBQ, kKeyBlock);
      for (int n0 = 0; n0 < nk; n0 += kKeyBlock) {
#pragma unroll
        for (int kb = 0; kb < 2; ++kb) {
          const uint32_t a0 = smem_u32(sQ + kb * kTileBytes);
          const uint32_t b0 = smem_u32(sKP + static_cast<size_t>(kb) * nkmax * 128 + n0 * 128);
#pragma unroll
          for (int k = 0; k < 4; ++k)
            mma_f16(tmem + static_cast<uint32_t>(n0), sw128_kmajor_desc(a0 + k * 32), sw128_kmajor_desc(b0 + k * 32),
                    idesc, (kb | k) != 0 ? 1u : 0u);
        }
      }
      mma_commit(mma_bar);
    }
  }

  // ---------------------------------------------------------------- 2. V^T tiles, in place
  bool ok = mbar_wait_warp(v_bar, 0, abort_flag, &g_attn_err);
  {
    // 128 threads per tile, four tiles at a time; thread: keys (t % 8) * 8 .. + 7
    // of the 64-key block, head dims ((t / 8) % 16) * 8 .. + 7
    const int tt = t & 127, kgl = tt & 7, dg = tt >> 3;
    const int half = dg >> 3, dc = dg & 7;  // which 8 KB half, 16-byte chunk in its 128-byte rows
    const int ntiles = nk / kKeyBlock;
    for (int j0 = 0; j0 < ntiles; j0 += kThreads / 128) {
      const int j = j0 + (t >> 7);
      uint8_t* tile = sVt + j * kTileBytes;
      uint4 in[8];
#pragma unroll
      for (int rr = 0; rr < 8; ++rr) {
        const int key = kgl * 8 + rr;  // row of the staged block
        in[rr] = (ok && j < ntiles && j * kKeyBlock + key < m)
                     ? *reinterpret_cast<const uint4*>(tile + half * 8192 + sw128_off(key, dc))
                     : make_uint4(0u, 0u, 0u, 0u);
      }
      __syncthreads();  // the blocks are in registers before any of them is overwritten
      if (j < ntiles) {
#pragma unroll
        for (int d = 0; d < 8; ++d) {
          const uint32_t sel = (d & 1) ? 0x7632u : 0x5410u;
          const int w = d >> 1;
          uint32_t o[4];
#pragma unroll
          for (int u = 0; u < 4; ++u) {
            const uint32_t a = w == 0 ? in[2 * u].x : w == 1 ? in[2 * u].y : w == 2 ? in[2 * u].z : in[2 * u].w;
            const uint32_t c = w == 0 ? in[2 * u + 1].x : w == 1 ? in[2 * u + 1].y : w == 2 ? in[2 * u + 1].z
                                                                                      : in[2 * u + 1].w;
            o[u] = __byte_perm(a, c, sel);
          }
          *reinterpret_cast<uint4*>(tile + sw128_off(dg * 8 + d, kgl)) = make_uint4(o[0], o[1], o[2], o[3]);
        }
      }
    }
  }

  // ---------------------------------------------------------------- 3. softmax rows -> P
  if (ok) ok = mbar_wait_warp(mma_bar, 0, abort_flag, &g_attn_err);
  tc_fence_after();
  const int lg = warp & (kLaneGroups - 1), cq = warp / kLaneGroups;  // lane group, first chunk
  const int row = lg * 32 + (t & 31);                                // query row of the block
  const int qpos = qb * kBQ + row;
  const int lim = min(qpos, m - 1);  // last key of this row
  const uint32_t trow = tmem + (static_cast<uint32_t>(lg * 32) << 16);
  // chunks of 32 columns the lane group's rows can see (the TMEM loads are
  // warp-wide, the causal limit differs by row)
  const int nch = min(qb * kBQ + lg * 32 + 31, m - 1) / 32 + 1;
  constexpr int kStep = kThreads / 32 / kLaneGroups;  // warps per lane group
  float l = 0.0f;
  if (ok) {
    float mx = -INFINITY;
    for (int c = cq; c < nch; c += kStep) {
      uint32_t r[32];
      tmem_ld_32x32b_x32(trow + static_cast<uint32_t>(c * 32), r);
      tmem_ld_wait();
#pragma unroll
      for (int e = 0; e < 32; ++e)
        if (c * 32 + e <= lim) mx = fmaxf(mx, __uint_as_float(r[e]));
    }
    red[cq * kBQ + row] = mx;
  }
  __syncthreads();
  if (ok) {
    float mx = red[row];
#pragma unroll
    for (int k = 1; k < kStep; ++k) mx = fmaxf(mx, red[k * kBQ + row]);
    const float off = mx * p.c2;
    for (int c = cq; c < nch; c += kStep) {
      uint32_t r[32];
      tmem_ld_32x32b_x32(trow + static_cast<uint32_t>(c * 32), r);
      tmem_ld_wait();
      uint32_t hp[16];
#pragma unroll
      for (int e = 0; e < 32; e += 2) {
        const int j = c * 32 + e;
        const float p0 = j <= lim ? exp2f(fmaf(__uint_as_float(r[e]), p.c2, -off)) : 0.0f;
        const float p1 = j + 1 <= lim ? exp2f(fmaf(__uint_as_float(r[e + 1]), p.c2, -off)) : 0.0f;
        l += p0;
        l += p1;
        const __half2 hh = __floats2half2_rn(p0, p1);
        hp[e >> 1] = *reinterpret_cast<const uint32_t*>(&hh);
      }
      // 32 keys = 4 chunks of 8 in the P tile of key block c / 2
      uint8_t* tile = sKP + (c >> 1) * kTileBytes;
      const int cc = (c & 1) * 4;
#pragma unroll
      for (int u = 0; u < 4; ++u)
        *reinterpret_cast<uint4*>(tile + sw128_off(row, cc + u)) =
            make_uint4(hp[4 * u], hp[4 * u + 1], hp[4 * u + 2], hp[4 * u + 3]);
    }
  }
  // P is zero in the chunks past the rows' causal limit
  for (int c = nch + cq; c < nk / 32; c += kStep) {
    uint8_t* tile = sKP + (c >> 1) * kTileBytes;
#pragma unroll
    for (int u = 0; u < 4; ++u)
      *reinterpret_cast<uint4*>(tile + sw128_off(row, (c & 1) * 4 + u)) = make_uint4(0u, 0u, 0u, 0u);
  }
  fence_proxy_async_smem();  // P and V^T (generic writes) -> the tensor cores
  tc_fence_before();
  __syncthreads();  // every warp has read the row maxima before they are overwritten
  red[cq * kBQ + row] = l;

  // ---------------------------------------------------------------- 4. O = P V
  if (t == 0 && ok && !*abort_flag) {
    tc_fence_after();
    constexpr uint32_t idesc = idesc_f16_f32(kBQ, kDH);
    for (int j = 0; j < nk / kKeyBlock; ++j) {
      const uint32_t a0 = smem_u32(sKP + j * kTileBytes);
      const uint32_t b0 = smem_u32(sVt + j * kTileBytes);
#pragma unroll
      for (int k = 0; k < 4; ++k)
        mma_f16(tmem, sw128_kmajor_desc(a0 + k * 32), sw128_kmajor_desc(b0 + k * 32), idesc, (j | k) != 0 ? 1u : 0u);
    }
    mma_commit(mma_bar);
  }
  __syncthreads();  // the row sums are in shared memory
  // ok is uniform across each warp (it comes from warp-wide waits): every
  // lane of a warp takes the same branch into the warp-wide wait
  if (ok) ok = mbar_wait_warp(mma_bar, 1, abort_flag, &g_attn_err);
  tc_fence_after();
  if (ok) {
    float sum = red[row];
#pragma unroll
    for (int k = 1; k < kStep; ++k) sum += red[k * kBQ + row];
    const float inv = 1.0f / sum;
    const int c0 = cq * 32;  // this warp's 32 head dimensions
    uint32_t r[32];
    tmem_ld_32x32b_x32(trow + static_cast<uint32_t>(c0), r);
    tmem_ld_wait();
    if (qpos < m) {
      __half* orow = p.o + (static_cast<size_t>(b) * m + qpos) * p.ldo + h * kDH + c0;
      uint32_t hv[16];
#pragma unroll
      for (int e = 0; e < 32; e += 2) {
        const __half2 hh = __floats2half2_rn(__uint_as_float(r[e]) * inv, __uint_as_float(r[e + 1]) * inv);
        hv[e >> 1] = *reinterpret_cast<const uint32_t*>(&hh);
      }
#pragma unroll
      for (int u = 0; u < 4; ++u)
        *reinterpret_cast<uint4*>(orow + 8 * u) = make_uint4(hv[4 * u], hv[4 * u + 1], hv[4 * u + 2], hv[4 * u + 3]);
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 0) tmem_dealloc(tmem, tmem_cols);
}

// 3-D map over fp16 rows [1][rows][cols] with row pitch ld elements; boxes of
// 64 columns (128 bytes, 128-byte swizzle) x box_rows rows.
bool make_rows_map(CUtensorMap* map, const uint16_t* base, int rows, int cols, long long ld, int box_rows) {
  auto enc = get_encode_fn();
  if (!enc) return false;
  cuuint64_t dims[3] = {static_cast<cuuint64_t>(cols), static_cast<cuuint64_t>(rows), 1};
  cuuint64_t strides[2] = {static_cast<cuuint64_t>(ld) * 2, static_cast<cuuint64_t>(ld) * 2 * rows};
  cuuint32_t box[3] = {64, static_cast<cuuint32_t>(box_rows), 1};
  cuuint32_t estr[3] = {1, 1, 1};
  return enc(map, CU_TENSOR_MAP_DATA_TYPE_FLOAT16, 3, const_cast<uint16_t*>(base), dims, strides, box, estr,
             CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
             CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

}  // namespace

size_t causal_attention_smem_bytes(int m) {
  const int nkmax = ((m + kKeyBlock - 1) / kKeyBlock) * kKeyBlock;
  return 1024 + 2 * kTileBytes + static_cast<size_t>(nkmax) * 512 + 64;
}

cudaError_t launch_causal_attention(const uint16_t* q, long long ldq, const uint16_t* k, long long ldk,
                                    const uint16_t* v, long long ldv, int B, int m, int H, int Hkv, uint16_t* o,
                                    long long ldo, cudaStream_t stream) {
  if (B <= 0) return cudaSuccess;
  const size_t smem = causal_attention_smem_bytes(m);
  static size_t smem_set = 0;
  if (smem > smem_set) {
    cudaError_t e = cudaFuncSetAttribute(causal_attention_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         static_cast<int>(causal_attention_smem_bytes(kAttnMaxLen)));
    if (e != cudaSuccess) return e;
    smem_set = causal_attention_smem_bytes(kAttnMaxLen);
  }
  CUtensorMap mq, mk, mv;
  if (!make_rows_map(&mq, q, B * m, H * kDH, ldq, kBQ)) return cudaErrorInvalidValue;
  if (!make_rows_map(&mk, k, B * m, Hkv * kDH, ldk, kKeyBlock)) return cudaErrorInvalidValue;
  if (!make_rows_map(&mv, v, B * m, Hkv * kDH, ldv, kKeyBlock)) return cudaErrorInvalidValue;
  AttnParams p;
  p.o = reinterpret_cast<__half*>(o);
  p.ldo = ldo;
  p.m = m;
  p.group = H / Hkv;
  p.nkmax = ((m + kKeyBlock - 1) / kKeyBlock) * kKeyBlock;
  p.c2 = 1.4426950408889634f / sqrtf(static_cast<float>(kDH));
  const dim3 grid((m + kBQ - 1) / kBQ, H, B);
  return launch_pdl(causal_attention_kernel, grid, dim3(kThreads), smem, stream, mq, mk, mv, p);
}

unsigned int attn_read_and_clear_error() {
  unsigned int v = 0, z = 0;
  cudaMemcpyFromSymbol(&v, g_attn_err, sizeof(v));
  cudaMemcpyToSymbol(g_attn_err, &z, sizeof(z));
  return v;
}

}  // namespace p4q
