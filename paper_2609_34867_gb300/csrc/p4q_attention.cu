// Causal softmax attention on the pruned sequence with FP16 keys and values
// (App. B: the language model's linears run in W4A4 while the key and value
// caches stay in FP16). Per sample of m positions and per head h:
//   o_i = sum_{j <= i} p_ij v_j,  p_i. = softmax_j(q_i . k_j / sqrt(d_h)),
// key/value head h / (H / H_kv).
//
// Work unit: one 128-query block of one head of one sample; it sees keys
// 0 .. 128 (qb + 1) - 1 (qb its block index), taken in chunks of 128 with an
// online softmax (running row maxima and sums). The (sample, head) pairs are
// taken in groups whose units fill about one wave of CTAs, so that the query
// blocks of a head run side by side and share its keys and values through
// L2; inside a group the longest units come first, and the waves are dealt
// to the persistent CTAs (one per unit of a group, at most one per SM) in
// alternating directions. Ten warps:
//   warp 0     loads by TMA: each unit's query tile, each chunk's keys and
//              values into two-stage rings (keys one chunk ahead of values;
//              a key stage is free once its S is computed, a value stage once
//              its P V is);
//   warp 1     issues the tensor-core MMAs (tcgen05 kind::f16, fp32
//              accumulators in TMEM): S = Q K^T of a chunk into one of two
//              S buffers (the next chunk's S before this chunk's P V inside
//              a unit), and O += P V with P read from TMEM and V read in
//              place as an MN-major operand (no transposed copy);
//   warps 2-9  two threads per query row (its TMEM lane), one per half of
//              the chunk's keys and of O's columns: the chunk's row maximum
//              (the halves meet in shared memory), p = 2^((s - m)
//              log2(e) / sqrt(d_h)) (0 past the causal limit on the diagonal
//              chunk) rounded to fp16 into TMEM over the chunk's S, and the
//              row sum. The reference maximum m of a row moves only when the
//              chunk's maximum exceeds it by more than 8 / (log2(e) /
//              sqrt(d_h)) (so p <= 2^8, exact in fp16's range), and then O
//              and the sum are rescaled by 2^((m_old - m_new) ...); the
//              softmax is the same for any reference. O is double-buffered:
//              a unit's O / sum -> fp16 runs after the next unit's first
//              chunk.
// Keys and rows past m read as zeros (3-D tensor maps over [B][m][cols]).
// Every wait of the pipeline polls the barrier and is bounded; a time-out
// sets the kernel's device error word.
#include <cuda_fp16.h>

#include <algorithm>

#include "p4q.h"
#include "p4q_device.cuh"
#include "p4q_internal.h"

namespace p4q {

__device__ unsigned int g_attn_err;

namespace {

constexpr int kBQ = 128;           // query rows per unit (TMEM lanes)
constexpr int kDH = 128;           // head dimension
constexpr int kChunk = 128;        // keys per chunk
constexpr int kThreads = 320;      // load warp, MMA warp, eight softmax warps
constexpr int kTileBytes = 16384;  // 128 rows x 128 bytes (64 fp16, 128-byte swizzle)

struct AttnParams {
  __half* o;
  long long ldo;
  long long hb;       // H * B (sample, head) pairs
  long long padded;   // units including the empty slots of the last group
  int m, H, group, nq, gsz;
  float c2;           // log2(e) / sqrt(d_h)
};

// Shared memory: two query buffers, two key stages, two value stages (two
// tiles each: head dims 0-63, 64-127), the row maxima / sums of the two
// halves of each row, barriers.
constexpr int kQBufs = 2;    // query buffers (units in flight)
constexpr int kKStages = 2;  // key stages
constexpr int kOffQ = 0;
constexpr int kOffK = kOffQ + 2 * kQBufs * kTileBytes;
constexpr int kOffV = kOffK + 2 * kKStages * kTileBytes;
constexpr int kOffRed = kOffV + 4 * kTileBytes;  // float [3 (chunk parity; row sums)][2 (half)][128]
constexpr int kOffBar = kOffRed + 6 * kBQ * 4;
constexpr int kNumBars = 18;
constexpr int kSmemBytes = 1024 + kOffBar + kNumBars * 8 + 16;
static_assert(kSmemBytes <= 232448, "one CTA per SM");
// TMEM columns: O buffers 0 .. and 128 .., S buffers 256 .. and 384 ..; a
// chunk's P (fp16 pairs, 64 columns) overwrites the first half of its S.
constexpr uint32_t kTmemCols = 512;
constexpr uint32_t kColS = 256;

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

// Instruction descriptor of kind::f16 with fp16 A and B and an fp32
// accumulator, for an M x N tile; A and B K-major (bit 16 set: B MN-major).
__host__ __device__ constexpr uint32_t idesc_f16_f32(int M, int N) {
  return (1u << 4)                                 // D format F32
         | (0u << 7) | (0u << 10)                  // A, B format F16
         | (static_cast<uint32_t>(N >> 3) << 17)   // N / 8
         | (static_cast<uint32_t>(M >> 4) << 24);  // M / 16
}

// A from TMEM (lanes = rows, two fp16 of K per column), B from shared memory.
__device__ __forceinline__ void mma_f16_ts(uint32_t d_tmem, uint32_t a_tmem, uint64_t b_desc, uint32_t idesc,
                                           uint32_t accumulate) {
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "setp.ne.b32 p, %4, 0;\n\t"
      "tcgen05.mma.cta_group::1.kind::f16 [%0], [%1], %2, %3, p;\n\t}\n" ::"r"(d_tmem),
      "r"(a_tmem), "l"(b_desc), "r"(idesc), "r"(accumulate)
      : "memory");
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

// Shared-memory descriptor of an MN-major operand in 128-byte swizzled atoms
// (8 rows of K x 64 fp16 along MN per 1024-byte atom, as a TMA box of 64
// columns writes them): atoms every 1024 bytes along K (stride offset) and
// every `mn_stride` bytes along MN (leading offset).
__device__ __forceinline__ uint64_t sw128_mnmajor_desc(uint32_t saddr, uint32_t mn_stride) {
  uint64_t d = 0;
  d |= static_cast<uint64_t>((saddr & 0x3FFFFu) >> 4);
  d |= static_cast<uint64_t>(mn_stride >> 4) << 16;
  d |= static_cast<uint64_t>(1024 >> 4) << 32;
  d |= static_cast<uint64_t>(1) << 46;
  d |= static_cast<uint64_t>(2) << 61;
  return d;
}

__device__ __forceinline__ float ex2_approx(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

// The units of one CTA in order, and their chunks: unit slot k of the CTA is
// u = k G + (k even ? x : G - 1 - x) (x its index, G the grid); unit u is,
// in group g = u / (nq gsz), block qb = nq - 1 - w / gsz of pair g gsz + w %
// gsz (w = u % (nq gsz)); slots whose pair is past H B are skipped. uq
// counts the CTA's units, c the unit's chunks (0 .. qb), j all its chunks.
struct ChunkIt {
  long long k, j;
  int uq, c, qb, h, b;
  bool valid;
  __device__ void seek(const AttnParams& p) {  // the first real unit from slot k on
    const long long G = gridDim.x, x = blockIdx.x;
    const long long per = static_cast<long long>(p.nq) * p.gsz;
    while (true) {
      const long long u = k * G + ((k & 1) ? (G - 1 - x) : x);
      if (u >= p.padded) {
        valid = false;
        return;
      }
      const long long g = u / per, w = u - g * per;
      const long long bh = g * p.gsz + w % p.gsz;
      if (bh < p.hb) {
        valid = true;
        qb = p.nq - 1 - static_cast<int>(w / p.gsz);
        h = static_cast<int>(bh % p.H);
        b = static_cast<int>(bh / p.H);
        return;
      }
      ++k;
    }
  }
  __device__ void start(const AttnParams& p) {
    k = 0;
    j = 0;
    uq = 0;
    c = 0;
    seek(p);
  }
  __device__ void next(const AttnParams& p) {
    ++j;
    if (++c > qb) {
      c = 0;
      ++uq;
      ++k;
      seek(p);
    }
  }
};

struct Bars {
  uint64_t q_full[kQBufs], q_empty[kQBufs], k_full[kKStages], k_empty[kKStages];
  uint64_t v_full[2], v_empty[2], s_full[2];
  uint64_t o_free[2];  // per O buffer: a unit's output has been read out
  uint64_t p_ready, pv_done, mma_done;
  uint32_t tmem_slot;
  int abort_flag;
};
static_assert(sizeof(Bars) <= kNumBars * 8 + 16, "barrier area");

__global__ void __launch_bounds__(kThreads, 1)
    causal_attention_kernel(const __grid_constant__ CUtensorMap tmQ, const __grid_constant__ CUtensorMap tmK,
                            const __grid_constant__ CUtensorMap tmV, const AttnParams p) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  Bars& br = *reinterpret_cast<Bars*>(smem + kOffBar);
  const int t = threadIdx.x, warp = t >> 5, lane = t & 31;
  volatile int* abort_flag = &br.abort_flag;

  if (t == 0) {
    for (int i = 0; i < kQBufs; ++i) {
      mbar_init(&br.q_full[i], 1);
      mbar_init(&br.q_empty[i], 1);
    }
    for (int i = 0; i < kKStages; ++i) {
      mbar_init(&br.k_full[i], 1);
      mbar_init(&br.k_empty[i], 1);
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(&br.v_full[i], 1);
      mbar_init(&br.v_empty[i], 1);
      mbar_init(&br.s_full[i], 1);
      mbar_init(&br.o_free[i], 8);
    }
    mbar_init(&br.p_ready, 8);
    mbar_init(&br.pv_done, 1);
    mbar_init(&br.mma_done, 1);
    br.abort_flag = 0;
    fence_barrier_init();
  }
  if (warp == 1) {
    tmem_alloc(&br.tmem_slot, kTmemCols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = br.tmem_slot;
  pdl_wait();  // q, k, v come from the previous kernel
  pdl_launch_dependents();

  if (warp == 0) {
    // ---------------------------------------------------------------- loads
    if (lane == 0) {
      tma_prefetch_desc(&tmQ);
      tma_prefetch_desc(&tmK);
      tma_prefetch_desc(&tmV);
      bool ok = true;
      long long k_issued = 0, v_issued = 0;
      int q_issued = 0;
      ChunkIt kit, vit;
      kit.start(p);
      vit.start(p);
      // keys of a chunk (and the unit's queries with its first chunk)
      auto load_k = [&](const ChunkIt& it) {
        const int hk = it.h / p.group;
        if (it.c == 0) {
          const int qbuf = it.uq % kQBufs;
          if (it.uq >= kQBufs)
            ok = ok && mbar_wait_spin(&br.q_empty[qbuf], ((it.uq / kQBufs) - 1) & 1, abort_flag, &g_attn_err);
          if (!ok) return;
          mbar_arrive_expect_tx(&br.q_full[qbuf], 2 * kTileBytes);
          for (int kb = 0; kb < 2; ++kb)
            tma_load_3d(&tmQ, &br.q_full[qbuf], smem + kOffQ + (2 * qbuf + kb) * kTileBytes, it.h * kDH + kb * 64,
                        it.qb * kBQ, it.b);
          ++q_issued;
        }
        const int st = static_cast<int>(it.j % kKStages);
        if (it.j >= kKStages)
          ok = ok && mbar_wait_spin(&br.k_empty[st], ((it.j / kKStages) - 1) & 1, abort_flag, &g_attn_err);
        if (!ok) return;
        mbar_arrive_expect_tx(&br.k_full[st], 2 * kTileBytes);
        for (int kb = 0; kb < 2; ++kb)
          tma_load_3d(&tmK, &br.k_full[st], smem + kOffK + (2 * st + kb) * kTileBytes, hk * kDH + kb * 64,
                      it.c * kChunk, it.b);
        ++k_issued;
      };
      auto load_v = [&](const ChunkIt& it) {
        const int st = static_cast<int>(it.j & 1);
        if (it.j >= 2) ok = ok && mbar_wait_spin(&br.v_empty[st], ((it.j >> 1) - 1) & 1, abort_flag, &g_attn_err);
        if (!ok) return;
        mbar_arrive_expect_tx(&br.v_full[st], 2 * kTileBytes);
        for (int kb = 0; kb < 2; ++kb)
          tma_load_3d(&tmV, &br.v_full[st], smem + kOffV + (2 * st + kb) * kTileBytes, (it.h / p.group) * kDH + kb * 64,
                      it.c * kChunk, it.b);
        ++v_issued;
      };
      if (kit.valid) {
        load_k(kit);
        kit.next(p);
      }
      while (ok && vit.valid) {
        if (kit.valid) {  // keys one chunk ahead of the values
          load_k(kit);
          kit.next(p);
        }
        if (ok) load_v(vit);
        vit.next(p);
      }
      // nothing of this CTA's loads may still be in flight when it exits
      volatile int never = 0;
      for (long long jj = k_issued - 1; jj >= 0 && jj >= k_issued - kKStages; --jj)
        mbar_wait(&br.k_full[jj % kKStages], (jj / kKStages) & 1, &never, &g_attn_err);
      for (long long jj = v_issued - 1; jj >= 0 && jj >= v_issued - 2; --jj)
        mbar_wait(&br.v_full[jj & 1], (jj >> 1) & 1, &never, &g_attn_err);
      for (int qq = q_issued - 1; qq >= 0 && qq >= q_issued - kQBufs; --qq)
        mbar_wait(&br.q_full[qq % kQBufs], (qq / kQBufs) & 1, &never, &g_attn_err);
    }
  } else if (warp == 1) {
    // ---------------------------------------------------------------- MMAs
    if (lane == 0) {
      bool ok = true;
      constexpr uint32_t idS = idesc_f16_f32(kBQ, kChunk);
      constexpr uint32_t idO = idesc_f16_f32(kBQ, kDH) | (1u << 16);  // B (V) MN-major
      ChunkIt sit, pit;
      sit.start(p);
      pit.start(p);
      // S = Q K^T of a chunk into S buffer j & 1. The buffer held the S, then
      // the P, of chunk j - 2, whose P V this thread issued earlier: the
      // tcgen05.mma operations of one thread run in issue order, so that P V
      // has read its P before this S overwrites it.
      auto issue_s = [&](const ChunkIt& it) {
        const int qbuf = it.uq % kQBufs, st = static_cast<int>(it.j & 1), ks = static_cast<int>(it.j % kKStages);
        if (it.c == 0) ok = ok && mbar_wait_spin(&br.q_full[qbuf], (it.uq / kQBufs) & 1, abort_flag, &g_attn_err);
        ok = ok && mbar_wait_spin(&br.k_full[ks], (it.j / kKStages) & 1, abort_flag, &g_attn_err);
        if (!ok) return;
        tc_fence_after();
        const uint32_t d = tmem + kColS + 128u * static_cast<uint32_t>(st);
#pragma unroll
        for (int kb = 0; kb < 2; ++kb) {
          const uint32_t a0 = smem_u32(smem + kOffQ + (2 * qbuf + kb) * kTileBytes);
          const uint32_t b0 = smem_u32(smem + kOffK + (2 * ks + kb) * kTileBytes);
#pragma unroll
          for (int k = 0; k < 4; ++k)
            mma_f16(d, sw128_kmajor_desc(a0 + 32 * k), sw128_kmajor_desc(b0 + 32 * k), idS, (kb | k) != 0 ? 1u : 0u);
        }
        mma_commit(&br.s_full[st]);
        mma_commit(&br.k_empty[ks]);
        if (it.c == it.qb) mma_commit(&br.q_empty[qbuf]);
      };
      if (sit.valid) {
        issue_s(sit);
        sit.next(p);
      }
      while (ok && pit.valid) {
        // inside a unit the next chunk's S goes before this chunk's P V; the
        // next unit's first S right after it
        const bool ahead = sit.valid && sit.uq == pit.uq;
        if (ahead) {
          issue_s(sit);
          sit.next(p);
        }
        ok = ok && mbar_wait_spin(&br.p_ready, pit.j & 1, abort_flag, &g_attn_err);
        // O buffer uq & 1 has been read out (unit uq - 2); one barrier per
        // buffer, so its phases cannot run two ahead of this wait
        if (pit.c == 0 && pit.uq >= 2)
          ok = ok && mbar_wait_spin(&br.o_free[pit.uq & 1], ((pit.uq >> 1) - 1) & 1, abort_flag, &g_attn_err);
        const int st = static_cast<int>(pit.j & 1);
        ok = ok && mbar_wait_spin(&br.v_full[st], (pit.j >> 1) & 1, abort_flag, &g_attn_err);
        if (!ok) break;
        tc_fence_after();
        const uint32_t d = tmem + 128u * static_cast<uint32_t>(pit.uq & 1);
#pragma unroll
        for (int kt = 0; kt < kChunk / 16; ++kt) {  // 16 keys per MMA: 8 P columns, 16 V rows
          const uint32_t bv = smem_u32(smem + kOffV + 2 * st * kTileBytes) + 2048 * kt;
          mma_f16_ts(d, tmem + kColS + 128u * static_cast<uint32_t>(st) + 8u * kt,
                     sw128_mnmajor_desc(bv, kTileBytes), idO, (pit.c > 0 || kt > 0) ? 1u : 0u);
        }
        mma_commit(&br.v_empty[st]);
        mma_commit(&br.pv_done);
        if (!ahead && sit.valid) {
          issue_s(sit);
          sit.next(p);
        }
        pit.next(p);
      }
      // every MMA of this CTA has completed before TMEM is released
      mma_commit(&br.mma_done);
      volatile int never = 0;
      mbar_wait(&br.mma_done, 0, &never, &g_attn_err);
    }
  } else {
    // ---------------------------------------------------------------- softmax and epilogue
    const int quad = warp & 3;             // TMEM lanes 32 quad .. + 31
    const int half = (warp - 2) >> 2;      // keys / O columns 64 half .. + 63
    const int r = quad * 32 + lane;        // query row of the unit
    const int rmax_warp = quad * 32 + 31;  // the warp's last row
    const uint32_t tl = tmem + (static_cast<uint32_t>(quad * 32) << 16);
    float* red = reinterpret_cast<float*>(smem + kOffRed);
    // O / sum -> fp16 of a finished unit, from O buffer ob (its last P V is done)
    int e_qb = 0, e_h = 0, e_b = 0, e_ob = 0;
    float e_l = 0.0f;
    bool pending = false;
    auto epilogue = [&](bool live) {
      float* rl = red + 4 * kBQ;  // row sums of the halves (rewritten one unit later, after
                                  // the partner has passed the chunk barriers in between)
      rl[half * kBQ + r] = e_l;
      named_bar_sync(1 + quad, 64);
      const float inv = 1.0f / (rl[r] + rl[kBQ + r]);
      const int qpos = e_qb * kBQ + r;
      __half* orow = p.o + (static_cast<size_t>(e_b) * p.m + qpos) * p.ldo + static_cast<size_t>(e_h) * kDH + 64 * half;
      if (live) {
#pragma unroll 1
        for (int oc = 0; oc < 2; ++oc) {
          uint32_t o[32];
          tmem_ld_32x32b_x32(tl + 128u * e_ob + 64u * half + 32u * oc, o);
          tmem_ld_wait();
          if (qpos < p.m) {
            uint32_t hv[16];
#pragma unroll
            for (int e = 0; e < 32; e += 2) {
              const __half2 hh = __floats2half2_rn(__uint_as_float(o[e]) * inv, __uint_as_float(o[e + 1]) * inv);
              hv[e >> 1] = *reinterpret_cast<const uint32_t*>(&hh);
            }
#pragma unroll
            for (int u4 = 0; u4 < 4; ++u4)
              *reinterpret_cast<uint4*>(orow + 32 * oc + 8 * u4) =
                  make_uint4(hv[4 * u4], hv[4 * u4 + 1], hv[4 * u4 + 2], hv[4 * u4 + 3]);
          }
        }
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&br.o_free[e_ob]);
    };
    // The two warps of a quad meet at a named barrier every chunk: after a
    // failed wait a warp keeps walking its chunks (no more waits, no TMEM
    // work) so that its partner is never left at a barrier.
    bool ok = true;
    ChunkIt it;
    it.start(p);
    float mrow = -INFINITY, l = 0.0f;
    for (; it.valid; it.next(p)) {
      const int st = static_cast<int>(it.j & 1);
      const uint32_t ts = tl + kColS + 128u * st;  // this chunk's S (then P)
      if (ok) ok = mbar_wait_spin_warp(&br.s_full[st], (it.j >> 1) & 1, abort_flag, &g_attn_err);
      tc_fence_after();
      uint32_t sv[2][32];
      if (ok) {
#pragma unroll
        for (int q2 = 0; q2 < 2; ++q2) tmem_ld_32x32b_x32(ts + 64u * half + 32u * q2, sv[q2]);
        tmem_ld_wait();
      } else {
#pragma unroll
        for (int q2 = 0; q2 < 2; ++q2)
#pragma unroll
          for (int e = 0; e < 32; ++e) sv[q2][e] = 0u;
      }
      const bool diag = it.c == it.qb;     // keys past the row are masked only here
      const int key0 = 64 * half;          // first key of this half in the chunk
      float m4[4] = {-INFINITY, -INFINITY, -INFINITY, -INFINITY};
#pragma unroll
      for (int e = 0; e < 64; ++e)
        if (!diag || key0 + e <= r) m4[e & 3] = fmaxf(m4[e & 3], __uint_as_float(sv[e >> 5][e & 31]));
      float* rd = red + (st * 2) * kBQ;    // [half][row] of this chunk parity
      rd[half * kBQ + r] = fmaxf(fmaxf(m4[0], m4[1]), fmaxf(m4[2], m4[3]));
      named_bar_sync(1 + quad, 64);        // both halves have their S in registers and their maxima out
      const float mx = fmaxf(rd[r], rd[kBQ + r]);
      if (it.c == 0) {
        mrow = -INFINITY;
        l = 0.0f;
      }
      // the row's reference maximum (finite: key 0 of the diagonal chunk is
      // always visible) moves only when the chunk's exceeds it by 2^8 in p
      const float mnew = (it.c == 0 || (mx - mrow) * p.c2 > 8.0f) ? fmaxf(mrow, mx) : mrow;
      const float alpha = (it.c == 0 || mnew == mrow) ? 1.0f : ex2_approx((mrow - mnew) * p.c2);
      const float off = mnew * p.c2;
      float l4[4] = {0.0f, 0.0f, 0.0f, 0.0f};
      uint32_t hp[32];
#pragma unroll
      for (int k8 = 0; k8 < 8; ++k8) {
        if (!diag || key0 + 8 * k8 <= rmax_warp) {  // uniform: some row of the warp sees the group
#pragma unroll
          for (int e2 = 0; e2 < 4; ++e2) {
            const int e = 8 * k8 + 2 * e2;
            float p0 = ex2_approx(fmaf(__uint_as_float(sv[e >> 5][e & 31]), p.c2, -off));
            float p1 = ex2_approx(fmaf(__uint_as_float(sv[(e + 1) >> 5][(e + 1) & 31]), p.c2, -off));
            if (diag) {
              p0 = key0 + e <= r ? p0 : 0.0f;
              p1 = key0 + e + 1 <= r ? p1 : 0.0f;
            }
            l4[e2] += p0 + p1;
            const __half2 hh = __floats2half2_rn(p0, p1);
            hp[4 * k8 + e2] = *reinterpret_cast<const uint32_t*>(&hh);
          }
        } else {
#pragma unroll
          for (int e2 = 0; e2 < 4; ++e2) hp[4 * k8 + e2] = 0u;
        }
      }
      l = l * alpha + ((l4[0] + l4[1]) + (l4[2] + l4[3]));
      // P over the first half of this chunk's S (both halves of every row
      // have loaded their S: the barrier above)
      if (ok) tmem_st_32x32b_x32(ts + 32u * half, hp);
      // O of the earlier chunks follows the new maximum, after their P V
      // (which also ends the previous unit, whose O is read out below)
      if (ok && it.j > 0) ok = mbar_wait_spin_warp(&br.pv_done, (it.j - 1) & 1, abort_flag, &g_attn_err);
      tc_fence_after();
      if (ok && it.c > 0 && __any_sync(0xFFFFFFFFu, alpha != 1.0f)) {
#pragma unroll 1
        for (int oc = 0; oc < 2; ++oc) {
          uint32_t o[32];
          const uint32_t ta = tl + 128u * (it.uq & 1) + 64u * half + 32u * oc;
          tmem_ld_32x32b_x32(ta, o);
          tmem_ld_wait();
#pragma unroll
          for (int e = 0; e < 32; ++e) o[e] = __float_as_uint(__uint_as_float(o[e]) * alpha);
          tmem_st_32x32b_x32(ta, o);
        }
      }
      tmem_st_wait();
      mrow = mnew;
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&br.p_ready);
      if (pending) {  // the previous unit's output, under this chunk's P V
        epilogue(ok);
        pending = false;
      }
      if (it.c == it.qb) {
        pending = true;
        e_qb = it.qb;
        e_h = it.h;
        e_b = it.b;
        e_ob = it.uq & 1;
        e_l = l;
      }
    }
    if (pending) {  // the last unit
      const long long jl = it.j - 1;
      if (ok && jl >= 0) ok = mbar_wait_spin_warp(&br.pv_done, jl & 1, abort_flag, &g_attn_err);
      tc_fence_after();
      epilogue(ok);
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 1) tmem_dealloc(tmem, kTmemCols);
}

// 3-D map over fp16 rows [B][m][cols] with row pitch ld elements (rows past m
// of a sample read as zeros); boxes of 64 columns (128 bytes, 128-byte
// swizzle) x 128 rows.
bool make_rows_map(CUtensorMap* map, const uint16_t* base, int B, int m, int cols, long long ld) {
  auto enc = get_encode_fn();
  if (!enc) return false;
  cuuint64_t dims[3] = {static_cast<cuuint64_t>(cols), static_cast<cuuint64_t>(m), static_cast<cuuint64_t>(B)};
  cuuint64_t strides[2] = {static_cast<cuuint64_t>(ld) * 2, static_cast<cuuint64_t>(ld) * 2 * m};
  cuuint32_t box[3] = {64, 128, 1};
  cuuint32_t estr[3] = {1, 1, 1};
  return enc(map, CU_TENSOR_MAP_DATA_TYPE_FLOAT16, 3, const_cast<uint16_t*>(base), dims, strides, box, estr,
             CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
             CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

int attn_sm_count() {
  int dev = 0, n = 0;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev);
  return n > 0 ? n : 1;
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
  if (!make_rows_map(&mq, q, B, m, H * kDH, ldq)) return cudaErrorInvalidValue;
  if (!make_rows_map(&mk, k, B, m, Hkv * kDH, ldk)) return cudaErrorInvalidValue;
  if (!make_rows_map(&mv, v, B, m, Hkv * kDH, ldv)) return cudaErrorInvalidValue;
  AttnParams p;
  p.o = reinterpret_cast<__half*>(o);
  p.ldo = ldo;
  p.m = m;
  p.H = H;
  p.group = H / Hkv;
  p.nq = (m + kBQ - 1) / kBQ;
  p.hb = static_cast<long long>(H) * B;
  p.c2 = 1.4426950408889634f / sqrtf(static_cast<float>(kDH));
  // (sample, head) pairs per group, and a grid of exactly one group's units
  // (at most one per SM): every wave is one group, and a CTA's blocks
  // alternate between qb and nq - 1 - qb (the waves' alternating
  // directions), so that the CTAs' chunk counts stay even
  p.gsz = static_cast<int>(std::max<long long>(1, std::min<long long>(p.hb, attn_sm_count() / p.nq)));
  p.padded = (p.hb + p.gsz - 1) / p.gsz * p.gsz * p.nq;
  const long long grid = static_cast<long long>(p.gsz) * p.nq;
  return launch_pdl(causal_attention_kernel, dim3(static_cast<unsigned>(grid)), dim3(kThreads),
                    static_cast<size_t>(kSmemBytes), stream, mq, mk, mv, p);
}

unsigned int attn_read_and_clear_error() {
  unsigned int v = 0, z = 0;
  cudaMemcpyFromSymbol(&v, g_attn_err, sizeof(v));
  cudaMemcpyToSymbol(g_attn_err, &z, sizeof(z));
  return v;
}

}  // namespace p4q
