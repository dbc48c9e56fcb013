// Stage 3 of the selector (Sec. 3.2, Eq. 4, visual diversity): greedy
// max-min selection on the cosines of fake-quantized tokens. With R the kept
// set (R0 after stages 1-2), m_i = max over r in R of cos(i, r) (-inf while R
// is empty); each of the K_d rounds keeps the free token with the smallest
// m (lower index on ties) and m absorbs its cosines.
//
// One CTA per image. The largest cosine of every token to R0 comes from the
// tensor-core GEMM before this kernel (its cosine-max epilogue, or a row pass
// over its int32 tiles; in Gram mode a row pass over the token-pair GEMM)
// as m. After that no cosine row of the whole image is ever formed. The kernel holds, for every free token, a
// lower bound of m (exact up to the first ex picks) and runs in phases:
//   1. pool: the 128 smallest free (bound, token) pairs (block radix select);
//      tau = the largest of them. Every token outside the pool has a pair
//      above tau, and its true pair is at least its bound's.
//   2. the pool's exact cosines: code dot products of the pool rows with the
//      pool rows and with every pick the pool's bounds have not seen yet, on
//      the tensor cores (tcgen05 kind::f8f6f4, M = 128 pool rows, N <= 256
//      columns per chunk, operand rows gathered from the expanded codes into
//      a 4-deep ring of shared-memory stages by cp.async in the
//      128-byte-swizzled K-major layout),
//      turned into Eq. 4 cosines in the epilogue: the pool block and, per
//      pool row, the largest cosine to those picks (the bound becomes m).
//   3. greedy rounds on the pool by the block (pool_rounds): a pool entry
//      whose pair is at most tau is below every token outside, so the
//      smallest such entry is the next pick, and runs of the next smallest
//      are picked together while no earlier pick raises them; their cosines
//      to the pool come from the block.
//   4. the pool's m go back to their tokens (exact up to the picks so far).
// A phase that picks nothing still makes its pool exact, so phases end.
#include <cuda_fp16.h>

#include "p4q.h"
#include "p4q_device.cuh"
#include "p4q_internal.h"
#include "p4q_rank.cuh"

namespace p4q {

__device__ unsigned int g_diverse_err;

namespace {

constexpr int kPool = 128;
constexpr int kPickMax = 64;  // picks confirmed per pool iteration at most
constexpr int kPoolPer = kPool / 32;
static_assert(kPoolPer == 4, "pool warp layout: four slots per lane");
constexpr int kArows = 128;   // pool rows per MMA (M = 128: the TMEM lanes)
constexpr int kBrows = 128;   // extra column rows per stage
constexpr int kBK = 128;      // bytes of K per stage (one 128-byte swizzle row)
constexpr int kStages = 4;    // k-blocks in flight: the gathered rows come at L2 latency
constexpr int kLag = 2;       // k-blocks a producer keeps loading before it hands one over
constexpr int kAbytes = kArows * kBK;
constexpr int kStageBytes = (kArows + kBrows) * kBK;
constexpr uint32_t kTmemCols = 256;

struct DivScratch {
  unsigned int hist[256];
  unsigned int wsum[32];
  int digit, above;
  int t, npool, tmin, nphase;
  unsigned long long tau;
  __align__(16) unsigned long long skey[kPool];  // pool rounds: (m, slot) keys of the certain entries
  int sorted[kPool];                    // pool rounds: slots of the certain entries in key order
  int L;                                // pool rounds: length of the confirmed prefix
  int ptok[kPool];                      // pool slot -> token (ascending)
  float pm[kPool];                      // m of the pool tokens (bound, then exact)
  unsigned int pmx[kPool];              // order key of the largest cosine to the pick columns
  int psum[kPool], pnorm[kPool];        // pool rows: sum of u, squared code norm
  float prs[kPool];                     // pool rows: rsqrtf of the squared code norm (0 for a zero row)
  int csum[kBrows], cnorm[kBrows];      // extra columns of the current chunk
  float crs[kBrows];                    // their rsqrtf norms (candidate path)
  unsigned int keptbits[P4Q_MAX_TOKENS / 32];
  int16_t list[P4Q_MAX_TOKENS];         // the greedy picks, in order
  signed char slotof[P4Q_MAX_TOKENS];   // token -> pool slot, -1 outside the pool
  int16_t candof[P4Q_MAX_TOKENS];       // token -> candidate index, -1 for the others
  int pci[kPool];                       // pool slot -> candidate index (-1: not a candidate)
  uint64_t bar_full[kStages];           // producer warps -> the stage is in shared memory
  uint64_t bar_empty[kStages];          // MMA commit -> the stage may be overwritten
  uint64_t bar_acc;                     // MMA commit -> the chunk's accumulator is complete
  uint64_t bar_done;                    // MMA commit at teardown -> nothing in flight
  uint32_t tmem_slot;
  volatile int abort_flag;
  __align__(16) float cp[kPool][kPool + 1]; // cos(ptok[i], ptok[j]) (Eq. 4, exact; padded: column writes)
};

__device__ __forceinline__ float order_key_float(uint32_t k) {
  return __uint_as_float((k & 0x80000000u) ? (k & 0x7FFFFFFFu) : ~k);
}

// Greedy rounds on the pool, by the whole block (thread i < 128 owns pool
// slot i), with exact m of the pool entries in s.pm. The next pick is the
// smallest free (m, token) pair. A pool entry is certain to be in order while
// its pair is at most tau (every token outside the pool is above tau and m
// only grows). Per iteration the certain entries are ranked by their pairs
// (each owner counts the smaller keys), giving c_0 < c_1 < ...; c_0 is the
// next pick, and c_a the pick after c_0 .. c_{a-1} whenever none of their
// cosines exceeds m(c_a) (nothing else can pass it: every other pair only
// grows). The pairs (b < a) are checked in parallel; the longest such
// prefix (at most kPickMax) is picked at once, the pool's m absorbs the
// picks' cosines, and the picks are appended to s.list. Ends when Kd picks
// are made or no entry is certain; s.t and s.pm hold the results.
template <int kThreads>
__device__ void pool_rounds(int npool, int Kd, DivScratch& s) {
  constexpr unsigned long long kNone = ~0ull;
  const int tid = threadIdx.x;
  const unsigned long long tau = s.tau;
  bool alive = tid < npool;
  while (true) {
    const int t = s.t;  // every thread has passed the barrier that published it
    if (t >= Kd) break;
    unsigned long long key = kNone;
    if (alive) {
      const unsigned long long pr = (static_cast<unsigned long long>(float_order_key(s.pm[tid])) << 32) | tid;
      if (pr <= tau) key = pr;
    }
    if (tid < kPool) s.skey[tid] = key;
    if (tid == 0) s.L = kPickMax;
    const int nc = __syncthreads_count(key != kNone);
    const int r = min(min(nc, Kd - t), kPickMax);
    if (r == 0) break;
    // rank of each certain entry among them (keys are unique: the slot is in the low bits)
    int rank = kPool;
    if (key != kNone) {
      rank = 0;
#pragma unroll 8
      for (int f = 0; f < kPool; f += 2) {
        const ulonglong2 kk = *reinterpret_cast<const ulonglong2*>(&s.skey[f]);
        rank += (kk.x < key ? 1 : 0) + (kk.y < key ? 1 : 0);
      }
      if (rank < r) s.sorted[rank] = tid;
    }
    __syncthreads();
    // pairs b < a < r: a violation (an earlier candidate raises c_a) ends the prefix at a
    const int npairs = r * (r - 1) / 2;
    for (int q = tid; q < npairs; q += kThreads) {
      int a2 = static_cast<int>((1.0f + sqrtf(1.0f + 8.0f * static_cast<float>(q))) * 0.5f);
      while (a2 * (a2 - 1) / 2 > q) --a2;
      while ((a2 + 1) * a2 / 2 <= q) ++a2;
      const int b2 = q - a2 * (a2 - 1) / 2;
      const int ca = s.sorted[a2];
      if (s.cp[s.sorted[b2]][ca] > s.pm[ca]) atomicMin(&s.L, a2);
    }
    __syncthreads();
    const int L = min(s.L, r);  // >= 1: c_0 never fails
    if (alive) {
      if (rank < L) {
        alive = false;
        const int tok = s.ptok[tid];
        s.list[t + rank] = static_cast<int16_t>(tok);
        atomicOr(&s.keptbits[tok >> 5], 1u << (tok & 31));
      } else {
        float m = s.pm[tid];
#pragma unroll 8
        for (int b2 = 0; b2 < L; ++b2) m = fmaxf(m, s.cp[s.sorted[b2]][tid]);
        s.pm[tid] = m;
      }
    }
    if (tid == 0) s.t = t + L;
    __syncthreads();
  }
}

// Arguments of one launch.
struct DivArgs {
  const uint32_t* kept12;  // [B, words] R0 as bits
  const float* m;          // [B, N] largest cosine to R0 (R0 > 0)
  const int32_t* cand;     // [B, C] candidates, ascending (nullptr: every token, C = N)
  const int32_t* candnorm; // [B, C]
  const float* cdots;      // [B, C, cpitch] their pairwise code dot products
  int C, cpitch;
  const uint8_t* vu;       // [B*N, d] expanded codes
  const int32_t* vsum;     // [B*N]
  const int32_t* vnorm;    // [B*N]
  int N, d, R0, K, Kd;
  int32_t* idx;            // [B, K]
};

template <int kThreads>
__global__ void __launch_bounds__(kThreads, 1) select_diverse_kernel(const DivArgs a) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* stages = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  DivScratch& s = *reinterpret_cast<DivScratch*>(stages + kStages * kStageBytes);
  constexpr int kWarps = kThreads / 32;
  const int b = blockIdx.x, N = a.N, d = a.d;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int tpg = ((N + kPer - 1) / kPer + 31) / 32 * 32;  // token owners (group 0)
  const bool g0 = threadIdx.x < tpg;
  const int base = kPer * threadIdx.x;
  const int words = (N + 31) / 32;
  const size_t row0 = static_cast<size_t>(b) * N;

  if (threadIdx.x == 0) {
    for (int i = 0; i < kStages; ++i) {
      mbar_init(&s.bar_full[i], kThreads / 32 - 1);
      mbar_init(&s.bar_empty[i], 1);
    }
    mbar_init(&s.bar_acc, 1);
    mbar_init(&s.bar_done, 1);
    s.abort_flag = 0;
    s.t = 0;
    s.nphase = 0;
    fence_barrier_init();
  }
  if (warp == 0) {
    tmem_alloc(&s.tmem_slot, kTmemCols);
    tmem_relinquish();
  }
  for (int i = threadIdx.x; i < N; i += kThreads) {
    s.slotof[i] = -1;
    s.candof[i] = -1;
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = s.tmem_slot;
  volatile int* abort_flag = &s.abort_flag;
  pdl_wait();  // R0 bits and maxima come from the kernels before
  pdl_launch_dependents();
  for (int w = threadIdx.x; w < words; w += kThreads) s.keptbits[w] = a.kept12[static_cast<size_t>(b) * words + w];
  __syncthreads();  // candof is cleared
  for (int c = threadIdx.x; c < a.C; c += kThreads)
    s.candof[a.cand ? a.cand[static_cast<size_t>(b) * a.C + c] : c] = static_cast<int16_t>(c);
  __syncthreads();

  bool kept[kPer];
  float m[kPer];
  int ex[kPer];  // m of the token is exact up to the first ex picks
#pragma unroll
  for (int e = 0; e < kPer; ++e) {
    const int i = base + e;
    kept[e] = g0 && i < N && ((s.keptbits[i >> 5] >> (i & 31)) & 1u);
    m[e] = -INFINITY;
    ex[e] = 0;
    if (g0 && i < N && !kept[e] && a.R0 > 0) m[e] = a.m[row0 + i];
  }
  const int KB = d / kBK;
  const int phase_limit = a.Kd * (N / kPool + 2) + 8;
  int g = 0;       // k-blocks staged so far (mbarrier phases of bar_full / bar_empty)
  int chunks = 0;  // accumulators completed so far (phases of bar_acc)
  uint32_t key[kPer];

  while (true) {
    __syncthreads();
    const int t = s.t;
    if (t >= a.Kd || s.abort_flag) break;
    if (threadIdx.x == 0 && ++s.nphase > phase_limit) {
      s.abort_flag = 1;
      atomicOr(&g_diverse_err, kErrTimeout);
    }
#pragma unroll
    for (int e = 0; e < kPer; ++e)
      if (g0 && base + e < N && ((s.keptbits[(base + e) >> 5] >> ((base + e) & 31)) & 1u)) kept[e] = true;
    // ---- 1. pool: the q smallest free (bound, token) pairs, in token order
    const int nfree = N - a.R0 - t;
    const int q = min(kPool, nfree);
    if (threadIdx.x == 0) s.tmin = t;
    int npool = 0;
    if (g0) {
      bool member[kPer];
#pragma unroll
      for (int e = 0; e < kPer; ++e) {
        member[e] = kept[e];
        key[e] = (base + e < N) ? ~float_order_key(m[e]) : 0u;
      }
      block_take_top(key, member, base, N, q, tpg, s);
      int cnt = 0, emin = t;
#pragma unroll
      for (int e = 0; e < kPer; ++e) {
        const bool in = base + e < N && member[e] && !kept[e];
        cnt += in ? 1 : 0;
        emin = in ? min(emin, ex[e]) : emin;
      }
      int pos = block_exclusive_scan(cnt, &npool, tpg, s);
#pragma unroll
      for (int e = 0; e < kPer; ++e) {
        if (base + e < N && member[e] && !kept[e]) {
          const int i = base + e;
          s.ptok[pos] = i;
          s.pm[pos] = m[e];
          s.pmx[pos] = 0u;  // below the key of every float
          s.psum[pos] = a.vsum[row0 + i];
          s.pnorm[pos] = a.vnorm[row0 + i];
          s.prs[pos] = s.pnorm[pos] > 0 ? rsqrtf(static_cast<float>(s.pnorm[pos])) : 0.0f;
          s.slotof[i] = static_cast<signed char>(pos);
          s.pci[pos] = s.candof[i];
          ++pos;
        }
      }
      if (emin < t) atomicMin(&s.tmin, emin);
      if (threadIdx.x == 0) s.npool = npool;
    }
    __syncthreads();
    npool = s.npool;
    const int tmin = s.tmin;
    const int ncp = t - tmin;  // picks whose cosines some pool bound has not seen
    // tau: the largest pool pair (everything certain when the pool holds every free token)
    if (warp == 0) {
      unsigned long long mx = 0;
#pragma unroll
      for (int k = 0; k < kPoolPer; ++k) {
        const int slot = kPoolPer * lane + k;
        if (slot < npool) {
          const unsigned long long pr = (static_cast<unsigned long long>(float_order_key(s.pm[slot])) << 32) | slot;
          mx = pr > mx ? pr : mx;
        }
      }
      const uint32_t thi = __reduce_max_sync(0xFFFFFFFFu, static_cast<uint32_t>(mx >> 32));
      const uint32_t tlo =
          __reduce_max_sync(0xFFFFFFFFu, static_cast<uint32_t>(mx >> 32) == thi ? static_cast<uint32_t>(mx) : 0u);
      if (lane == 0) s.tau = (q >= nfree) ? ~0ull : ((static_cast<unsigned long long>(thi) << 32) | tlo);
    }
    // ---- 2. the pool's exact dot products with the pool and with the picks
    // its bounds have not seen: from the candidates' dot products when every
    // one of those tokens is a candidate, else on the tensor cores here
    bool mine_ok = true;
    for (int r = threadIdx.x; r < npool + ncp; r += kThreads) {
      const int tok = r < npool ? s.ptok[r] : s.list[tmin + r - npool];
      mine_ok = mine_ok && s.candof[tok] >= 0;
    }
    const bool from_cand = __syncthreads_and(mine_ok) != 0;
    if (from_cand) {
      const float* cd = a.cdots + static_cast<size_t>(b) * a.C * a.cpitch;
      // the pool block, one warp per row, four columns per lane in flight
      for (int e = warp; e < npool; e += kWarps) {
        const float* row = cd + static_cast<size_t>(s.pci[e]) * a.cpitch;
        float v[kPoolPer];
#pragma unroll
        for (int k = 0; k < kPoolPer; ++k) {
          const int f = lane + 32 * k;
          v[k] = f < npool ? __ldg(row + s.pci[f]) : 0.0f;
        }
        const int ne = s.pnorm[e];
        // the block is symmetric: each pair once (f >= e), written both ways
#pragma unroll
        for (int k = 0; k < kPoolPer; ++k) {
          const int f = lane + 32 * k;
          if (f < npool && f >= e) {
            const float c = code_cosine(static_cast<int>(v[k]), ne, s.pnorm[f]);
            s.cp[e][f] = c;
            s.cp[f][e] = c;
          }
        }
      }
      // per pool row: the largest cosine to the unseen picks (chunks of 128
      // picks with their candidate index and norms in shared memory),
      // approximate first, then exact for the columns near it
      const int32_t* cn = a.candnorm + static_cast<size_t>(b) * a.C;
      for (int c0 = 0; c0 < ncp; c0 += kBrows) {
        const int nc2 = min(kBrows, ncp - c0);
        __syncthreads();  // the previous chunk's column data is no longer read
        for (int c = threadIdx.x; c < nc2; c += kThreads) {
          const int cj = s.candof[s.list[tmin + c0 + c]];
          const int nj = cn[cj];
          s.csum[c] = cj;  // candidate index of the column
          s.cnorm[c] = nj;
          s.crs[c] = nj > 0 ? rsqrtf(static_cast<float>(nj)) : 0.0f;
        }
        __syncthreads();
        for (int e = warp; e < npool; e += kWarps) {
          const float* row = cd + static_cast<size_t>(s.pci[e]) * a.cpitch;
          float v[kBrows / 32];
#pragma unroll
          for (int k = 0; k < kBrows / 32; ++k) {
            const int c = lane + 32 * k;
            v[k] = c < nc2 ? __ldg(row + s.csum[c]) : 0.0f;
          }
          float amax = -INFINITY;
#pragma unroll
          for (int k = 0; k < kBrows / 32; ++k) {
            const int c = lane + 32 * k;
            if (c < nc2) amax = fmaxf(amax, v[k] * s.prs[e] * s.crs[c]);
          }
#pragma unroll
          for (int o = 16; o > 0; o >>= 1) amax = fmaxf(amax, __shfl_xor_sync(0xFFFFFFFFu, amax, o));
          float emax = -INFINITY;
#pragma unroll
          for (int k = 0; k < kBrows / 32; ++k) {
            const int c = lane + 32 * k;
            if (c < nc2 && v[k] * s.prs[e] * s.crs[c] >= amax - kCosMargin)
              emax = fmaxf(emax, code_cosine(static_cast<int>(v[k]), s.pnorm[e], s.cnorm[c]));
          }
#pragma unroll
          for (int o = 16; o > 0; o >>= 1) emax = fmaxf(emax, __shfl_xor_sync(0xFFFFFFFFu, emax, o));
          if (lane == 0) s.pmx[e] = max(s.pmx[e], float_order_key(emax));
        }
      }
      __syncthreads();
    } else {
    // the rows this phase reads, toward L2 ahead of the staged loads
    for (int r = threadIdx.x; r < npool + ncp; r += kThreads) {
      const int tok = r < npool ? s.ptok[r] : s.list[tmin + r - npool];
      prefetch_l2_bulk(a.vu + (row0 + tok) * d, static_cast<uint32_t>(d));
    }
    // chunk 0: columns = the 128 pool rows (the A stage itself) + up to 128 picks;
    // chunk c >= 1: up to 128 further picks.
    const int extra0 = min(ncp, kArows);
    const int nchunks = 1 + (ncp - extra0 + kBrows - 1) / kBrows;
    for (int ch = 0; ch < nchunks; ++ch) {
      const int pick0 = (ch == 0) ? tmin : tmin + extra0 + (ch - 1) * kBrows;  // first pick column of the chunk
      const int nextra = (ch == 0) ? extra0 : min(kBrows, ncp - extra0 - (ch - 1) * kBrows);
      const int ncol = (ch == 0) ? (extra0 > 0 ? kArows + ((nextra + 15) & ~15) : ((npool + 15) & ~15))
                                 : ((nextra + 15) & ~15);
      for (int c = threadIdx.x; c < nextra; c += kThreads) {
        const int tok = s.list[pick0 + c];
        s.csum[c] = a.vsum[row0 + tok];
        s.cnorm[c] = a.vnorm[row0 + tok];
      }
      const int items = (npool + nextra) * (kBK / 16);
      if (warp == 0) {
        // MMA issuer: each stage once its producers have arrived on full[st]
        if (lane == 0) {
          const uint32_t idesc = idesc_e4m3_f32(kArows, ncol);
          for (int kb = 0; kb < KB; ++kb, ++g) {
            const int st = g % kStages;
            if (!mbar_wait_spin(&s.bar_full[st], (g / kStages) & 1, abort_flag, &g_diverse_err)) continue;
            tc_fence_after();
            const uint32_t a0 = smem_u32(stages + st * kStageBytes);
            const uint32_t b0 = (ch == 0) ? a0 : a0 + kAbytes;
#pragma unroll
            for (int k = 0; k < kBK / 32; ++k)
              mma_f8f6f4(tmem, sw128_kmajor_desc(a0 + 32 * k), sw128_kmajor_desc(b0 + 32 * k), idesc,
                         (kb > 0 || k > 0) ? 1u : 0u);
            mma_commit(&s.bar_empty[st]);
          }
          mma_commit(&s.bar_acc);
        } else {
          g += KB;
        }
        __syncwarp();
      } else {
        // producers: warps 1.. gather the k-block's 16-byte row chunks by
        // cp.async; k-block kb is handed over (wait, proxy fence, arrive) kLag
        // k-blocks later, so kLag loads per thread stay in flight
        const int pt = threadIdx.x - 32, np = kThreads - 32;
        for (int kb = 0; kb < KB + kLag; ++kb) {
          if (kb < KB) {
            const int st = (g + kb) % kStages;
            if (g + kb >= kStages) {
              if (lane == 0)
                mbar_wait_spin(&s.bar_empty[st], (((g + kb) / kStages) - 1) & 1, abort_flag, &g_diverse_err);
              __syncwarp();
            }
            const uint32_t sbase = smem_u32(stages + st * kStageBytes);
            for (int it = pt; it < items; it += np) {
              // pool rows at stage rows 0.., extra columns at stage rows 128.. (the B region)
              const int r = it >> 3, c16 = it & 7;
              const bool pool_row = r < npool;
              const int tok = pool_row ? s.ptok[r] : s.list[pick0 + r - npool];
              const int srow = pool_row ? r : kArows + (r - npool);
              const uint8_t* src = a.vu + (row0 + tok) * d + kb * kBK + c16 * 16;
              cp_async16(sbase + srow * kBK + ((c16 ^ (srow & 7)) << 4), src);
            }
          }
          cp_async_commit();  // empty groups past KB keep the accounting uniform
          const int kc = kb - kLag;
          if (kc >= 0) {
            cp_async_wait<kLag>();
            fence_proxy_async_smem();
            __syncwarp();
            if (lane == 0) mbar_arrive(&s.bar_full[(g + kc) % kStages]);
          }
        }
        g += KB;
      }
      // epilogue: TMEM lanes = pool rows, 16-column groups spread over the warps
      if (lane == 0 && !*abort_flag) mbar_wait(&s.bar_acc, chunks & 1, abort_flag, &g_diverse_err);
      __syncwarp();
      ++chunks;
      tc_fence_after();
      {
        const int qd = warp & 3;
        const int e = 32 * qd + lane;
        const bool erow = e < npool;
        const float corr = erow ? static_cast<float>(64 * d - 8 * s.psum[e]) : 0.0f;
        const int ne = erow ? s.pnorm[e] : 0;
        // pool columns: every cosine, exactly (the block); pick columns: the
        // largest approximate cosine, then the exact cosine of the columns
        // near it (two passes over TMEM)
        float amax = -INFINITY, emax = -INFINITY;
        const int g_first = (ch == 0) ? kArows / 16 : 0;  // first group of pick columns
#pragma unroll 1
        for (int pass = 0; pass < 2; ++pass) {
#pragma unroll 1
          for (int grp = warp >> 2; grp < ncol / 16; grp += kWarps / 4) {  // the same groups in both passes
            if (pass == 1 && grp < g_first) continue;
            uint32_t v[16];
            tmem_ld_32x32b_x16(tmem + (static_cast<uint32_t>(32 * qd) << 16) + 16 * grp, v);
            tmem_ld_wait();
            if (!erow) continue;
            if (grp < g_first) {  // pool columns (pass 0 only)
#pragma unroll
              for (int i = 0; i < 16; ++i) {
                const int slot = 16 * grp + i;
                if (slot < npool) {
                  const int dot = __float2int_rn(__fmaf_rn(__uint_as_float(v[i]), 262144.0f,
                                                           corr - 8.0f * static_cast<float>(s.psum[slot])));
                  s.cp[slot][e] = code_cosine(dot, ne, s.pnorm[slot]);  // the block is symmetric
                }
              }
            } else {
#pragma unroll
              for (int i = 0; i < 16; ++i) {
                const int ci = 16 * grp + i - (ch == 0 ? kArows : 0);
                if (ci < nextra) {
                  const int dot = __float2int_rn(__fmaf_rn(__uint_as_float(v[i]), 262144.0f,
                                                           corr - 8.0f * static_cast<float>(s.csum[ci])));
                  const float ap = cos_approx(dot, ne, s.cnorm[ci]);
                  if (pass == 0) {
                    amax = fmaxf(amax, ap);
                  } else if (ap >= amax - kCosMargin) {
                    emax = fmaxf(emax, code_cosine(dot, ne, s.cnorm[ci]));
                  }
                }
              }
            }
          }
        }
        if (erow && emax > -INFINITY) atomicMax(&s.pmx[e], float_order_key(emax));
      }
      tc_fence_before();
      __syncthreads();
    }
    }  // tensor-core path
    // the bounds of the pool become m
    if (threadIdx.x < npool && s.pmx[threadIdx.x] != 0u)
      s.pm[threadIdx.x] = fmaxf(s.pm[threadIdx.x], order_key_float(s.pmx[threadIdx.x]));
    __syncthreads();
    // ---- 3. greedy rounds on the pool
    if (!s.abort_flag) pool_rounds<kThreads>(npool, a.Kd, s);
    __syncthreads();
    // ---- 4. exact m back to the pool's tokens
    const int tn = s.t;
    if (g0) {
#pragma unroll
      for (int e = 0; e < kPer; ++e) {
        const int i = base + e;
        if (i < N && s.slotof[i] >= 0) {
          const int slot = s.slotof[i];
          if ((s.keptbits[i >> 5] >> (i & 31)) & 1u) {
            kept[e] = true;
          } else {
            m[e] = s.pm[slot];
            ex[e] = tn;
          }
          s.slotof[i] = -1;
        }
      }
    }
  }
  // Output: the kept set in ascending index order.
  if (g0) {
    int cnt = 0;
#pragma unroll
    for (int e = 0; e < kPer; ++e)
      cnt += (base + e < N && ((s.keptbits[(base + e) >> 5] >> ((base + e) & 31)) & 1u)) ? 1 : 0;
    int total;
    int pos = block_exclusive_scan(cnt, &total, tpg, s);
#pragma unroll
    for (int e = 0; e < kPer; ++e)
      if (base + e < N && ((s.keptbits[(base + e) >> 5] >> ((base + e) & 31)) & 1u) && pos < a.K)
        a.idx[static_cast<size_t>(b) * a.K + pos++] = base + e;
  }
  // Teardown: every MMA this CTA issued has completed (a commit after the last
  // one, waited for with a bound) before the accumulator is released.
  if (threadIdx.x == 0) {
    mma_commit(&s.bar_done);
    int fresh = 0;
    mbar_wait(&s.bar_done, 0, reinterpret_cast<volatile int*>(&fresh), &g_diverse_err, 100000000ull);
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 0) {
    tc_fence_after();
    tmem_dealloc(tmem, kTmemCols);
  }
}

constexpr size_t kDivSmem = 1024 + kStages * kStageBytes + sizeof(DivScratch);
static_assert(kDivSmem <= 232448, "shared memory budget");

}  // namespace

cudaError_t launch_select_diverse(const SelectPlan& p, const SelectWorkspace& ws, int32_t* idx, cudaStream_t stream) {
  if (p.Kd <= 0) return cudaSuccess;
  DivArgs a;
  a.kept12 = ws.kept12;
  a.m = ws.m;
  a.cand = ws.gram ? nullptr : ws.cand;
  a.candnorm = ws.gram ? ws.vnorm : ws.candnorm;  // Gram mode: candidate c is token c
  a.cdots = ws.cdots;
  a.C = ws.C;
  a.cpitch = ws.cpitch;
  a.vu = ws.vu;
  a.vsum = ws.vsum;
  a.vnorm = ws.vnorm;
  a.N = p.N;
  a.d = p.d;
  a.R0 = p.Kq + p.Ks;
  a.K = p.K;
  a.Kd = p.Kd;
  a.idx = idx;
  const int tpg = ((p.N + kPer - 1) / kPer + 31) / 32 * 32;
  auto go = [&](auto kern, int threads) -> cudaError_t {
    static bool attr_set = false;  // one flag per instantiation
    (void)attr_set;
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(kDivSmem));
    if (e != cudaSuccess) return e;
    return launch_pdl(kern, dim3(p.B), dim3(threads), kDivSmem, stream, a);
  };
  if (tpg <= 512) return go(select_diverse_kernel<512>, 512);
  if (tpg <= 768) return go(select_diverse_kernel<768>, 768);
  return go(select_diverse_kernel<1024>, 1024);
}

unsigned int diverse_read_and_clear_error() {
  unsigned int v = 0, z = 0;
  cudaMemcpyFromSymbol(&v, g_diverse_err, sizeof(v));
  cudaMemcpyToSymbol(g_diverse_err, &z, sizeof(z));
  return v;
}

}  // namespace p4q
