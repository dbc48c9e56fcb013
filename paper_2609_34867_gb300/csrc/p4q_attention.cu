// Causal softmax attention on the pruned sequence with FP16 keys and values
// (App. B: the language model's linears run in W4A4 while the key and value
// caches stay in FP16). Per sample of m positions and per head h:
//   o_i = sum_{j <= i} p_ij v_j,  p_i. = softmax_j(q_i . k_j / sqrt(d_h)),
// key/value head h / (H / H_kv).
//
// One CTA per (128-query block, head, sample), 8 warps, two CTAs per SM:
// warp w reads TMEM lanes 32 (w % 4) .. + 31 (query rows) and takes every
// second 32-column chunk from chunk w / 4 on (keys for S, head dimensions
// for O). The keys the block can see (rounded up to 64) are taken 128 at a
// time, with an online softmax (running row maxima and sums):
//   1. thread 0 loads the query block once, and per key chunk the keys and
//      values by TMA into 128-byte swizzled tiles (after the previous chunk's
//      P V has released them), and issues S = Q K^T on the tensor cores
//      (tcgen05 kind::f16, N = the chunk's keys, fp32 accumulators in TMEM
//      columns 128 ..);
//   2. every thread takes an 8 x 8 block of the staged values into registers
//      and, after a block-wide barrier, writes it back transposed, so that
//      each 64-key tile becomes K-major V^T (keys at or past m are zero);
//   3. the row maxima of the four warps sharing the rows meet in shared
//      memory; with the chunk's maximum folded into the running one (m_new),
//      p = 2^((s - m_new) log2(e) / sqrt(d_h)) (0 past the causal limit) goes
//      to fp16 K-major P tiles in the space the keys used, the partial sums
//      are scaled by 2^((m_old - m_new) ...) and grow by p, and so is the
//      accumulated O (TMEM columns 0 .. 127, read, scaled and written back
//      when a row's maximum moved);
//   4. thread 0 issues O += P V^T. After the last chunk each warp scales its
//      32 columns of O by 1 / sum and stores fp16.
// One chunk (a block that sees at most 128 keys) is a plain two-pass
// softmax. Every wait is bounded; a time-out sets the kernel's device error
// word.
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
// 128 keys per chunk and 8 warps: 99 KB of shared memory, 256 TMEM columns
// and 28 K registers per CTA, so that two CTAs share an SM and one's softmax
// overlaps the other's loads and MMAs.
constexpr int kChunk = 128;     // keys per chunk (S columns in TMEM)
constexpr int kThreads = 256;
constexpr int kLaneGroups = 4;     // warps w and w + 4k share TMEM lanes 32 (w % 4) ..
constexpr int kTileBytes = 16384;  // 128 rows x 128 bytes

struct AttnParams {
  __half* o;
  long long ldo;
  int m, group;
  float c2;  // log2(e) / sqrt(d_h)
};

// Shared memory: query tiles, K (then P) tiles of one chunk, V^T tiles of one
// chunk, the row reductions, barriers.
constexpr int kOffQ = 0;
constexpr int kOffKP = 2 * kTileBytes;
constexpr int kOffVt = kOffKP + kChunk * 256;
constexpr int kOffRed = kOffVt + kChunk * 256;
constexpr int kOffBar = kOffRed + 4 * kBQ * 4;
constexpr int kSmemBytes = 1024 + kOffBar + 64;
constexpr uint32_t kTmemCols = 128 + kChunk;  // O: columns 0 .. 127, S: 128 .. 128 + kChunk - 1
static_assert(kTmemCols == 256 || kTmemCols == 512, "TMEM allocations are powers of two");

__device__ __forceinline__ void tmem_st_32x32b_x32(uint32_t taddr, const uint32_t (&r)[32]) {
  asm volatile(
      "tcgen05.st.sync.aligned.32x32b.x32.b32 [%0], "
      "{%1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, %15, %16, "
      "%17, %18, %19, %20, %21, %22, %23, %24, %25, %26, %27, %28, %29, %30, %31, %32};" ::"r"(taddr),
      "r"(r[0]), "r"(r[1]), "r"(r[2]), "r"(r[3]), "r"(r[4]), "r"(r[5]), "r"(r[6]), "r"(r[7]), "r"(r[8]),
      "r"(r[9]), "r"(r[10]), "r"(r[11]), "r"(r[12]), "r"(r[13]), "r"(r[14]), "r"(r[15]), "r"(r[16]), "r"(r[17]),
      "r"(r[18]), "r"(r[19]), "r"(r[20]), "r"(r[21]), "r"(r[22]), "r"(r[23]), "r"(r[24]), "r"(r[25]), "r"(r[26]),
      "r"(r[27]), "r"(r[28]), "r"(r[29]), "r"(r[30]), "r"(r[31])
      : "memory");
}

__device__ __forceinline__ void tmem_st_wait() { asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory"); }

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

__global__ void __launch_bounds__(kThreads, 2)
    causal_attention_kernel(const __grid_constant__ CUtensorMap tmQ, const __grid_constant__ CUtensorMap tmK,
                            const __grid_constant__ CUtensorMap tmV, const AttnParams p) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint8_t* sQ = smem + kOffQ;    // 2 tiles: head dims 0-63, 64-127
  uint8_t* sKP = smem + kOffKP;  // K: 2 x [kChunk x 128 B]; then P tiles
  uint8_t* sVt = smem + kOffVt;  // staged V, then V^T tiles, one per 64 keys
  float* red = reinterpret_cast<float*>(smem + kOffRed);  // [4][128] partial row maxima, then sums
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + kOffBar);
  uint64_t* q_bar = bars;      // query tiles in
  uint64_t* k_bar = bars + 1;  // a chunk's keys in
  uint64_t* v_bar = bars + 2;  // a chunk's values in
  uint64_t* s_bar = bars + 3;  // a chunk's S = Q K^T done
  uint64_t* o_bar = bars + 4;  // a chunk's O += P V^T done
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + 5);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(bars + 6);

  const int qb = blockIdx.x, h = blockIdx.y, b = blockIdx.z;
  const int hk = h / p.group;
  const int t = threadIdx.x, warp = t >> 5;
  const int m = p.m;
  const int last_key = min(m, (qb + 1) * kBQ) - 1;                   // the block's last visible key
  const int nk = ((last_key + kKeyBlock) / kKeyBlock) * kKeyBlock;  // keys loaded, multiple of 64
  const int nchunks = (nk + kChunk - 1) / kChunk;

  if (t == 0) {
    for (int i = 0; i < 5; ++i) mbar_init(bars + i, 1);
    *abort_flag = 0;
    fence_barrier_init();
  }
  if (warp == 0) {
    tmem_alloc(tmem_slot, kTmemCols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  pdl_wait();
  pdl_launch_dependents();

  const int lg = warp & (kLaneGroups - 1), cq = warp / kLaneGroups;  // lane group, first 32-column chunk
  const int row = lg * 32 + (t & 31);                                // query row of the block
  const int qpos = qb * kBQ + row;
  const int lim = min(qpos, m - 1);                                  // last key of this row
  const int lim_lg = min(qb * kBQ + lg * 32 + 31, m - 1);           // last key any row of the lane group sees
  const uint32_t trow = tmem + (static_cast<uint32_t>(lg * 32) << 16);
  constexpr int kStep = kThreads / 32 / kLaneGroups;  // warps per lane group
  constexpr uint32_t kS = 128;                        // first S column

  bool pok = true;  // thread 0's producer path
  bool ok = true;   // uniform across each warp (it comes from warp-wide waits)
  float mrow = -INFINITY, lpart = 0.0f;
  if (t == 0) {
    tma_prefetch_desc(&tmQ);
    tma_prefetch_desc(&tmK);
    tma_prefetch_desc(&tmV);
    mbar_arrive_expect_tx(q_bar, static_cast<uint32_t>(2 * kTileBytes));
#pragma unroll
    for (int kb = 0; kb < 2; ++kb)
      tma_load_3d(&tmQ, q_bar, sQ + kb * kTileBytes, h * kDH + kb * 64, b * m + qb * kBQ, 0);
  }
  for (int c = 0; c < nchunks; ++c) {
    const int k0 = c * kChunk;
    const int nc = min(kChunk, nk - k0);  // keys of this chunk, a multiple of 64
    // ---------------------------------------------------------------- 1. loads and S = Q K^T
    if (t == 0 && pok) {
      if (c > 0) pok = mbar_wait(o_bar, (c - 1) & 1, abort_flag, &g_attn_err);  // buffers released
      if (pok) {
        mbar_arrive_expect_tx(v_bar, static_cast<uint32_t>(nc * 256));
        // values of keys k0 + 64 j .. + 63 -> tile j: dims 0-63 in its first 8 KB, 64-127 in the second
        for (int r0 = 0; r0 < nc; r0 += kKeyBlock)
          for (int kb = 0; kb < 2; ++kb)
            tma_load_3d(&tmV, v_bar, sVt + (r0 / kKeyBlock) * kTileBytes + kb * 8192, hk * kDH + kb * 64,
                        b * m + k0 + r0, 0);
        mbar_arrive_expect_tx(k_bar, static_cast<uint32_t>(nc * 256));
        for (int kb = 0; kb < 2; ++kb)
          for (int r0 = 0; r0 < nc; r0 += kKeyBlock)
            tma_load_3d(&tmK, k_bar, sKP + kb * (kChunk * 128) + r0 * 128, hk * kDH + kb * 64, b * m + k0 + r0, 0);
        if (c == 0) pok = mbar_wait(q_bar, 0, abort_flag, &g_attn_err);
        if (pok) pok = mbar_wait(k_bar, c & 1, abort_flag, &g_attn_err);
      }
      if (pok) {
        tc_fence_after();
        // one MMA per 16 head dimensions covers the whole chunk (N = nc keys)
        const uint32_t idesc = idesc_f16_f32(kBQ, nc);
#pragma unroll
        for (int kb = 0; kb < 2; ++kb) {
          const uint32_t a0 = smem_u32(sQ + kb * kTileBytes);
          const uint32_t b0 = smem_u32(sKP + kb * (kChunk * 128));
#pragma unroll
          for (int k = 0; k < 4; ++k)
            mma_f16(tmem + kS, sw128_kmajor_desc(a0 + k * 32), sw128_kmajor_desc(b0 + k * 32), idesc,
                    (kb | k) != 0 ? 1u : 0u);
        }
        mma_commit(s_bar);
      }
    }

    // ---------------------------------------------------------------- 2. V^T tiles, in place
    if (ok) ok = mbar_wait_warp(v_bar, c & 1, abort_flag, &g_attn_err);
    {
      // 128 threads per tile, four tiles at a time; thread: keys (t % 8) * 8 .. + 7
      // of the 64-key block, head dims ((t / 8) % 16) * 8 .. + 7
      const int tt = t & 127, kgl = tt & 7, dg = tt >> 3;
      const int half = dg >> 3, dc = dg & 7;  // which 8 KB half, 16-byte chunk in its 128-byte rows
      const int ntiles = nc / kKeyBlock;
      for (int j0 = 0; j0 < ntiles; j0 += kThreads / 128) {
        const int j = j0 + (t >> 7);
        uint8_t* tile = sVt + j * kTileBytes;
        uint4 in[8];
#pragma unroll
        for (int rr = 0; rr < 8; ++rr) {
          const int key = kgl * 8 + rr;  // row of the staged block
          in[rr] = (ok && j < ntiles && k0 + j * kKeyBlock + key < m)
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
              const uint32_t e2 = w == 0 ? in[2 * u + 1].x : w == 1 ? in[2 * u + 1].y : w == 2 ? in[2 * u + 1].z
                                                                                         : in[2 * u + 1].w;
              o[u] = __byte_perm(a, e2, sel);
            }
            *reinterpret_cast<uint4*>(tile + sw128_off(dg * 8 + d, kgl)) = make_uint4(o[0], o[1], o[2], o[3]);
          }
        }
      }
    }

    // ---------------------------------------------------------------- 3. softmax of the chunk -> P
    if (ok) ok = mbar_wait_warp(s_bar, c & 1, abort_flag, &g_attn_err);
    if (ok && c > 0) ok = mbar_wait_warp(o_bar, (c - 1) & 1, abort_flag, &g_attn_err);  // O is settled
    tc_fence_after();
    // 32-column chunks of this key chunk that the lane group's rows can see
    const int nch = min(nc, max(0, lim_lg + 1 - k0) + 31) / 32;
    float mx = -INFINITY;
    if (ok) {
      for (int cc = cq; cc < nch; cc += kStep) {
        uint32_t r[32];
        tmem_ld_32x32b_x32(trow + kS + static_cast<uint32_t>(cc * 32), r);
        tmem_ld_wait();
#pragma unroll
        for (int e = 0; e < 32; ++e)
          if (k0 + cc * 32 + e <= lim) mx = fmaxf(mx, __uint_as_float(r[e]));
      }
    }
    red[cq * kBQ + row] = mx;
    __syncthreads();
    if (ok) {
      float mc = red[row];
#pragma unroll
      for (int k = 1; k < kStep; ++k) mc = fmaxf(mc, red[k * kBQ + row]);
      const float mnew = fmaxf(mrow, mc);  // finite: chunk 0 holds key 0 of every row
      const float alpha = c > 0 ? exp2f((mrow - mnew) * p.c2) : 1.0f;
      const float off = mnew * p.c2;
      lpart *= alpha;
      for (int cc = cq; cc < nch; cc += kStep) {
        uint32_t r[32];
        tmem_ld_32x32b_x32(trow + kS + static_cast<uint32_t>(cc * 32), r);
        tmem_ld_wait();
        uint32_t hp[16];
#pragma unroll
        for (int e = 0; e < 32; e += 2) {
          const int j = k0 + cc * 32 + e;
          const float p0 = j <= lim ? exp2f(fmaf(__uint_as_float(r[e]), p.c2, -off)) : 0.0f;
          const float p1 = j + 1 <= lim ? exp2f(fmaf(__uint_as_float(r[e + 1]), p.c2, -off)) : 0.0f;
          lpart += p0;
          lpart += p1;
          const __half2 hh = __floats2half2_rn(p0, p1);
          hp[e >> 1] = *reinterpret_cast<const uint32_t*>(&hh);
        }
        // 32 keys = 4 chunks of 8 in the P tile of key block cc / 2
        uint8_t* tile = sKP + (cc >> 1) * kTileBytes;
#pragma unroll
        for (int u = 0; u < 4; ++u)
          *reinterpret_cast<uint4*>(tile + sw128_off(row, (cc & 1) * 4 + u)) =
              make_uint4(hp[4 * u], hp[4 * u + 1], hp[4 * u + 2], hp[4 * u + 3]);
      }
      // O accumulated over the earlier chunks follows the new maximum (this
      // warp's 32-column chunks of its lane group's rows)
      if (c > 0 && __any_sync(0xFFFFFFFFu, alpha != 1.0f)) {
        for (int oc = cq; oc < kDH / 32; oc += kStep) {
          uint32_t r[32];
          tmem_ld_32x32b_x32(trow + static_cast<uint32_t>(oc * 32), r);
          tmem_ld_wait();
#pragma unroll
          for (int e = 0; e < 32; ++e) r[e] = __float_as_uint(__uint_as_float(r[e]) * alpha);
          tmem_st_32x32b_x32(trow + static_cast<uint32_t>(oc * 32), r);
        }
        tmem_st_wait();
      }
      mrow = mnew;
    }
    // P is zero in the 32-key chunks past the rows' causal limit
    for (int cc = nch + cq; cc < nc / 32; cc += kStep) {
      uint8_t* tile = sKP + (cc >> 1) * kTileBytes;
#pragma unroll
      for (int u = 0; u < 4; ++u)
        *reinterpret_cast<uint4*>(tile + sw128_off(row, (cc & 1) * 4 + u)) = make_uint4(0u, 0u, 0u, 0u);
    }
    fence_proxy_async_smem();  // P and V^T (generic writes) -> the tensor cores
    tc_fence_before();
    __syncthreads();  // P, V^T and O settled; every warp has read the row maxima

    // ---------------------------------------------------------------- 4. O += P V^T
    if (t == 0 && pok && !*abort_flag) {
      tc_fence_after();
      constexpr uint32_t idesc = idesc_f16_f32(kBQ, kDH);
      for (int j = 0; j < nc / kKeyBlock; ++j) {
        const uint32_t a0 = smem_u32(sKP + j * kTileBytes);
        const uint32_t b0 = smem_u32(sVt + j * kTileBytes);
#pragma unroll
        for (int k = 0; k < 4; ++k)
          mma_f16(tmem, sw128_kmajor_desc(a0 + k * 32), sw128_kmajor_desc(b0 + k * 32), idesc,
                  (c | j | k) != 0 ? 1u : 0u);
      }
      mma_commit(o_bar);
    }
  }

  // ---------------------------------------------------------------- epilogue
  red[cq * kBQ + row] = lpart;
  __syncthreads();  // the partial row sums are in shared memory
  if (ok) ok = mbar_wait_warp(o_bar, (nchunks - 1) & 1, abort_flag, &g_attn_err);
  tc_fence_after();
  if (ok) {
    float sum = red[row];
#pragma unroll
    for (int k = 1; k < kStep; ++k) sum += red[k * kBQ + row];
    const float inv = 1.0f / sum;
    for (int c0 = cq * 32; c0 < kDH; c0 += kStep * 32) {  // this warp's 32-column chunks of head dimensions
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
          *reinterpret_cast<uint4*>(orow + 8 * u) =
              make_uint4(hv[4 * u], hv[4 * u + 1], hv[4 * u + 2], hv[4 * u + 3]);
      }
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 0) tmem_dealloc(tmem, kTmemCols);
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

size_t causal_attention_smem_bytes(int) { return kSmemBytes; }

cudaError_t launch_causal_attention(const uint16_t* q, long long ldq, const uint16_t* k, long long ldk,
                                    const uint16_t* v, long long ldv, int B, int m, int H, int Hkv, uint16_t* o,
                                    long long ldo, cudaStream_t stream) {
  if (B <= 0) return cudaSuccess;
  static bool attr_set = false;
  if (!attr_set) {
    cudaError_t e = cudaFuncSetAttribute(causal_attention_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         kSmemBytes);
    if (e != cudaSuccess) return e;
    attr_set = true;
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
  p.c2 = 1.4426950408889634f / sqrtf(static_cast<float>(kDH));
  const dim3 grid((m + kBQ - 1) / kBQ, H, B);
  return launch_pdl(causal_attention_kernel, grid, dim3(kThreads), static_cast<size_t>(kSmemBytes), stream, mq, mk,
                    mv, p);
}

unsigned int attn_read_and_clear_error() {
  unsigned int v = 0, z = 0;
  cudaMemcpyFromSymbol(&v, g_attn_err, sizeof(v));
  cudaMemcpyToSymbol(g_attn_err, &z, sizeof(z));
  return v;
}

}  // namespace p4q
