// Quantization-aware visual-token selector (Sec. 3.2, Eq. 4 of the paper).
//
// Inputs are the fake-quantized copies produced by the per-row quantizer:
// packed INT4 codes and the squared code norm of every visual token and every
// concept embedding. The cosine of two fake-quantized rows is evaluated on
// their codes (the positive per-row scales cancel):
//   cos(a, b) = (float)<c_a, c_b> / sqrtf((float)|c_a|^2 * (float)|c_b|^2)
// with every operation rounded to fp32 in that order, and 0 when a norm is 0.
//
// Kernels:
//   query_scores_kernel   one warp per visual token: signed integer dot
//                         products (dp4a on sign-extended nibbles) with the J
//                         concept codes, then the cosine per concept.
//   select_stages_kernel  one CTA per image, one thread per 4 tokens: stage 1 (per-concept
//                         top quota), stage 2 (CLS-saliency top K_s), stage 3
//                         (greedy max-min diversity on the cosine matrix of
//                         the image, computed beforehand on the tensor cores),
//                         then the kept set in ascending order.
// Every ranking orders by (score, lower token index first).
#include <cuda_fp16.h>

#include <algorithm>

#include "p4q.h"
#include "p4q_device.cuh"
#include "p4q_internal.h"

namespace p4q {
namespace {


__device__ __forceinline__ float code_cosine(int dot, int na, int nb) {
  if (na == 0 || nb == 0) return 0.0f;
  return __fdiv_rn(static_cast<float>(dot), __fsqrt_rn(__fmul_rn(static_cast<float>(na), static_cast<float>(nb))));
}

constexpr int kScoreWarps = 8;

// Four two's complement nibbles (the even or odd codes of a packed word,
// already moved to the low nibble of each byte) sign-extended to bytes.
__device__ __forceinline__ int sext_nibbles(uint32_t n) {
  return static_cast<int>((n & 0x0F0F0F0Fu) | ((n & 0x08080808u) * 0x1Eu));
}

// scores[b, j, i] = cos(concept j of image b, token i of image b). One CTA
// per kScoreWarps tokens of one image, one warp per token (many warps in
// flight: the kernel is latency-bound): the image's J concept codes are
// staged in shared memory, every lane loads 16-byte chunks of the token's
// packed codes and sign-extends each chunk once for all J concepts (dp4a on
// the sign-extended nibbles); lane j then finishes the cosine of concept j.
// kJ bounds J (the concept loops unroll to kJ: a small kJ keeps the code in
// the instruction cache).
template <int kJ>
__global__ void __launch_bounds__(kScoreWarps * 32)
    query_scores_kernel(const uint8_t* __restrict__ vcodes, const int32_t* __restrict__ vnorm,
                        const uint8_t* __restrict__ qcodes, const int32_t* __restrict__ qnorm, int B, int N, int d,
                        int J, float* __restrict__ scores) {
  pdl_wait();
  pdl_launch_dependents();
  extern __shared__ uint4 qs[];  // [J][d/32] chunks of 32 packed codes
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int b = blockIdx.y, i = blockIdx.x * kScoreWarps + warp;
  const int nvec = d >> 5;
  const uint4* tq = reinterpret_cast<const uint4*>(qcodes + static_cast<size_t>(b) * J * (d >> 1));
  const uint4* tv = reinterpret_cast<const uint4*>(vcodes + (static_cast<size_t>(b) * N + (i < N ? i : 0)) * (d >> 1));
  uint4 x[4];  // the first chunks of the token, loaded before the barrier
#pragma unroll
  for (int u = 0; u < 4; ++u) x[u] = (i < N && u * 32 + lane < nvec) ? __ldg(tv + u * 32 + lane) : make_uint4(0u, 0u, 0u, 0u);
  for (int c = threadIdx.x; c < J * nvec; c += blockDim.x) qs[c] = tq[c];
  __syncthreads();
  if (i >= N) return;
  int acc[kJ];
#pragma unroll
  for (int j = 0; j < kJ; ++j) acc[j] = 0;
  for (int c0 = 0; c0 < nvec; c0 += 4 * 32) {
    if (c0 > 0) {
#pragma unroll
      for (int u = 0; u < 4; ++u) {
        const int c = c0 + u * 32 + lane;
        x[u] = c < nvec ? __ldg(tv + c) : make_uint4(0u, 0u, 0u, 0u);
      }
    }
#pragma unroll
    for (int u = 0; u < 4; ++u) {
      const int c = c0 + u * 32 + lane;
      if (c >= nvec) continue;
      int e[4][2];  // sign-extended nibbles of the chunk: [word][low / high]
      const uint32_t w[4] = {x[u].x, x[u].y, x[u].z, x[u].w};
#pragma unroll
      for (int k = 0; k < 4; ++k) {
        e[k][0] = sext_nibbles(w[k]);
        e[k][1] = sext_nibbles(w[k] >> 4);
      }
#pragma unroll
      for (int j = 0; j < kJ; ++j) {
        if (j < J) {
          const uint4 y = qs[j * nvec + c];
          const uint32_t wy[4] = {y.x, y.y, y.z, y.w};
#pragma unroll
          for (int k = 0; k < 4; ++k)
            acc[j] = __dp4a(e[k][1], sext_nibbles(wy[k] >> 4), __dp4a(e[k][0], sext_nibbles(wy[k]), acc[j]));
        }
      }
    }
  }
  const int nv = vnorm[static_cast<size_t>(b) * N + i];
#pragma unroll
  for (int j = 0; j < kJ; ++j) {
    if (j < J) {
      const int dot = __reduce_add_sync(0xFFFFFFFFu, acc[j]);
      if (lane == j) scores[(static_cast<size_t>(b) * J + j) * N + i] = code_cosine(dot, qnorm[b * J + j], nv);
    }
  }
}

constexpr int kSelThreads = 1024;  // upper bound on the block
// Smaller blocks get more registers per thread: 512 threads for N <= 2048,
// 768 for N <= 3072, 1024 above.
constexpr int kSelThreadsSmall = 512, kSelThreadsMid = 768;
constexpr int kPer = 4;  // tokens per thread of group 0: token i = kPer * threadIdx.x + e
// Diversity stage: a pool of the kPool smallest free (m, token) pairs is
// iterated by one warp (kPool / 32 entries per lane) with the pool's cosine
// block in shared memory; at most kPick picks per iteration.
constexpr int kPool = 128, kPick = 16;
constexpr int kPoolPer = kPool / 32;
static_assert(kPoolPer == 4, "pool warp layout: four slots per lane");

struct BlockScratch {
  unsigned int hist[256];
  unsigned int wsum[32];
  int digit, above;
  int t, npend;                              // greedy picks so far; pending rows in list
  __align__(16) int pick[kPick];             // pool slots of this iteration's candidates, ascending
  int ptok[kPool];                           // pool slot -> token (ascending)
  float pm[kPool];                           // m of the pool tokens when the pool was built
  unsigned int keptbits[P4Q_MAX_TOKENS / 32];
  int list[P4Q_MAX_TOKENS];                  // rows still to apply to m (the kept set, then picks)
  __align__(16) float part[P4Q_MAX_TOKENS];  // partial maxima of the row groups other than group 0
  int slotof[P4Q_MAX_TOKENS];                // token -> pool slot, -1 outside the pool
  __align__(16) float cp[kPool][kPool];      // cos(ptok[i], ptok[j])
};

// Barrier of the first nt threads of the block (group 0, the token owners);
// the other row groups do not take part in the rankings.
__device__ __forceinline__ void group_sync(int nt) { named_bar_sync(1, static_cast<uint32_t>(nt)); }

// Exclusive prefix sum of per-thread counts over the first nt threads (thread order).
template <class Scratch>
__device__ int block_exclusive_scan(int v, int* total, int nt, Scratch& s) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  int x = v;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const int y = __shfl_up_sync(0xFFFFFFFFu, x, o);
    if (lane >= o) x += y;
  }
  if (lane == 31) s.wsum[warp] = x;
  group_sync(nt);
  if (warp == 0) {
    int w = lane < (nt >> 5) ? s.wsum[lane] : 0;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int y = __shfl_up_sync(0xFFFFFFFFu, w, o);
      if (lane >= o) w += y;
    }
    s.wsum[lane] = w;  // inclusive
  }
  group_sync(nt);
  const int before = (warp ? s.wsum[warp - 1] : 0) + x - v;
  *total = s.wsum[(nt >> 5) - 1];
  group_sync(nt);
  return before;
}

// Marks as kept the q free tokens with the largest keys (keys are the
// order-preserving images of fp32 scores; ties go to the lower token index).
// Radix select, 8 bits per pass, from the most significant byte; the
// histogram updates are aggregated per warp over equal digits, since scores
// of similar magnitude share their leading bytes.
template <class Scratch>
__device__ void block_take_top(const uint32_t (&key)[kPer], bool (&kept)[kPer], int base, int N, int q, int nt,
                               Scratch& s) {
  if (q <= 0) return;
  const int lane = threadIdx.x & 31;
  uint32_t prefix = 0, mask = 0;
  int need = q;
  for (int pass = 0; pass < 4; ++pass) {
    const int shift = 24 - 8 * pass;
    for (int h = threadIdx.x; h < 256; h += nt) s.hist[h] = 0;
    group_sync(nt);
#pragma unroll
    for (int e = 0; e < kPer; ++e) {
      const bool live = (base + e < N) && !kept[e] && (key[e] & mask) == prefix;
      const uint32_t dig = live ? ((key[e] >> shift) & 255u) : 256u;  // 256: not counted
      const unsigned peers = __match_any_sync(0xFFFFFFFFu, dig);
      if (live && (__ffs(peers) - 1) == lane) atomicAdd(&s.hist[dig], static_cast<unsigned>(__popc(peers)));
    }
    group_sync(nt);
    if (threadIdx.x < 32) {
      // lane l owns digits [8l, 8l+8); find the digit where the count from the top reaches need
      unsigned int c[8], own = 0;
#pragma unroll
      for (int k = 0; k < 8; ++k) {
        c[k] = s.hist[8 * lane + k];
        own += c[k];
      }
      unsigned int x = own;
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const unsigned int y = __shfl_down_sync(0xFFFFFFFFu, x, o);
        if (lane + o < 32) x += y;
      }
      const unsigned int above = x - own;  // sum over lanes > lane
      if (above < static_cast<unsigned>(need) && above + own >= static_cast<unsigned>(need)) {
        unsigned int acc = above;
        for (int k = 7; k >= 0; --k) {
          if (acc + c[k] >= static_cast<unsigned>(need)) {
            s.digit = 8 * lane + k;
            s.above = static_cast<int>(acc);
            break;
          }
          acc += c[k];
        }
      }
    }
    group_sync(nt);
    need -= s.above;
    prefix |= static_cast<uint32_t>(s.digit) << shift;
    mask |= 255u << shift;
    group_sync(nt);
  }
  // keys > prefix are taken; among keys == prefix the first `need` in index order
  int eq = 0;
#pragma unroll
  for (int e = 0; e < kPer; ++e)
    if (base + e < N && !kept[e] && key[e] == prefix) ++eq;
  int total;
  int rank = block_exclusive_scan(eq, &total, nt, s);
#pragma unroll
  for (int e = 0; e < kPer; ++e) {
    if (base + e < N && !kept[e]) {
      if (key[e] > prefix) {
        kept[e] = true;
      } else if (key[e] == prefix) {
        if (rank < need) kept[e] = true;
        ++rank;
      }
    }
  }
  group_sync(nt);
}

// Sorts four 64-bit values ascending (five compare-exchanges).
__device__ __forceinline__ void sort4(unsigned long long (&h)[kPoolPer]) {
  auto cx = [](unsigned long long& x, unsigned long long& y) {
    const unsigned long long lo = x < y ? x : y, hi = x < y ? y : x;
    x = lo;
    y = hi;
  };
  cx(h[0], h[1]);
  cx(h[2], h[3]);
  cx(h[0], h[2]);
  cx(h[1], h[3]);
  cx(h[1], h[2]);
}

// m <- max(m, row r of the image's cosine matrix) for the n rows listed in
// s.list, on all row groups of the block: group g takes chunks of eight rows
// g, g + groups, ...; every thread loads 16 bytes per row (its group-0
// thread's four tokens), so the loads of different groups overlap (one SM
// keeps few row loads of one warp in flight). Group 0 then merges the other
// groups' partial maxima. Ends with the block synchronized.
__device__ void apply_rows(float (&m)[kPer], const float* __restrict__ G, int gp, int N, int n, int tpg, int groups,
                           BlockScratch& s) {
  const int g = threadIdx.x / tpg;
  const int tb = kPer * (threadIdx.x - g * tpg);  // first token of this thread's slice
  float p[kPer];
#pragma unroll
  for (int e = 0; e < kPer; ++e) p[e] = -INFINITY;
  if (tb < N) {  // tb + kPer <= gp: the 16-byte load stays inside the row's pitch
    for (int j0 = 8 * g; j0 < n; j0 += 8 * groups) {
      float4 v[8];
#pragma unroll
      for (int u = 0; u < 8; ++u)
        v[u] = (j0 + u < n) ? *reinterpret_cast<const float4*>(G + static_cast<size_t>(s.list[j0 + u]) * gp + tb)
                            : make_float4(-INFINITY, -INFINITY, -INFINITY, -INFINITY);
#pragma unroll
      for (int u = 0; u < 8; ++u) {
        p[0] = fmaxf(p[0], v[u].x); p[1] = fmaxf(p[1], v[u].y);
        p[2] = fmaxf(p[2], v[u].z); p[3] = fmaxf(p[3], v[u].w);
      }
    }
    if (g > 0) *reinterpret_cast<float4*>(&s.part[(g - 1) * kPer * tpg + tb]) = make_float4(p[0], p[1], p[2], p[3]);
  }
  __syncthreads();
  if (g == 0 && tb < N) {
#pragma unroll
    for (int e = 0; e < kPer; ++e) m[e] = fmaxf(m[e], p[e]);
    for (int h = 1; h < groups; ++h) {
      const float4 q = *reinterpret_cast<const float4*>(&s.part[(h - 1) * kPer * tpg + tb]);
      m[0] = fmaxf(m[0], q.x); m[1] = fmaxf(m[1], q.y); m[2] = fmaxf(m[2], q.z); m[3] = fmaxf(m[3], q.w);
    }
  }
  __syncthreads();
}

// One phase of greedy rounds on the pool, by warp 0 (lane l holds slots
// 4l .. 4l + 3, in token order). The next pick is the smallest free
// (m, token) pair. A pool entry is certain to be in order while its pair is
// at most tau, the largest pair at the pool's construction: every token
// outside the pool was above tau then and m only grows. Per iteration the r
// smallest certain entries c_0 < c_1 < ... are taken by r rounds of a warp
// minimum; c_0 is the next pick, and c_a the pick after c_0 .. c_{a-1}
// whenever none of their cosines exceeds m(c_a) (nothing else can pass it).
// The longest such prefix is picked, the pool's m absorbs the picks' cosines,
// and the picked tokens are appended to s.list as rows still to apply to the
// tokens outside the pool. Ends when Kd picks are made or no entry is
// certain; s.t and s.npend hold the counts.
__device__ void pool_rounds(int npool, int Kd, BlockScratch& s) {
  const int lane = threadIdx.x & 31;
  const unsigned int lanes_below = (1u << lane) - 1u;
  constexpr unsigned long long kNone = ~0ull;
  float pm[kPoolPer];
  unsigned int alive = 0;
  unsigned long long mx = 0;
#pragma unroll
  for (int k = 0; k < kPoolPer; ++k) {
    const int slot = kPoolPer * lane + k;
    pm[k] = slot < npool ? s.pm[slot] : 0.0f;
    if (slot < npool) {
      alive |= 1u << k;
      const unsigned long long pr = (static_cast<unsigned long long>(float_order_key(pm[k])) << 32) | slot;
      mx = pr > mx ? pr : mx;
    }
  }
  const uint32_t thi = __reduce_max_sync(0xFFFFFFFFu, static_cast<uint32_t>(mx >> 32));
  const uint32_t tlo = __reduce_max_sync(0xFFFFFFFFu, static_cast<uint32_t>(mx >> 32) == thi ? static_cast<uint32_t>(mx) : 0u);
  const unsigned long long tau = (static_cast<unsigned long long>(thi) << 32) | tlo;
  int t = s.t, npend = 0;
  while (t < Kd) {
    unsigned long long h[kPoolPer];
    int nv = 0;
#pragma unroll
    for (int k = 0; k < kPoolPer; ++k) {
      const unsigned long long pr =
          (static_cast<unsigned long long>(float_order_key(pm[k])) << 32) | (kPoolPer * lane + k);
      h[k] = ((alive >> k) & 1u) && pr <= tau ? pr : kNone;
      nv += h[k] != kNone;
    }
    nv = __reduce_add_sync(0xFFFFFFFFu, nv);
    const int r = min(min(kPick, Kd - t), nv);
    if (r == 0) break;
    sort4(h);
    // The lane's sorted entries as 32-bit keys (the pair order is the key
    // order, ties between lanes resolving to the lower lane) and their slots
    // as a queue of 2-bit indices into the lane's four slots.
    uint32_t hk[kPoolPer];
    uint32_t perm = 0;
#pragma unroll
    for (int k = 0; k < kPoolPer; ++k) {
      hk[k] = static_cast<uint32_t>(h[k] >> 32);
      perm |= (static_cast<uint32_t>(h[k]) & 3u) << (2 * k);
    }
    // r rounds of the warp minimum (branch-free: r is uniform over the warp,
    // later rounds change nothing); a lane records the rounds of its pops
    uint32_t rks = 0, pks = 0;
    int np = 0;
#pragma unroll
    for (int a = 0; a < kPick; ++a) {
      const uint32_t wk = __reduce_min_sync(0xFFFFFFFFu, hk[0]);
      const unsigned int tied = __ballot_sync(0xFFFFFFFFu, hk[0] == wk);
      const bool mine = a < r && hk[0] == wk && (tied & lanes_below) == 0u;
      if (mine) {
        s.pick[a] = kPoolPer * lane + static_cast<int>(perm & 3u);
        rks |= static_cast<uint32_t>(a) << (4 * np);
        pks |= (perm & 3u) << (2 * np);
        ++np;
        perm >>= 2;
#pragma unroll
        for (int k = 0; k + 1 < kPoolPer; ++k) hk[k] = hk[k + 1];
        hk[kPoolPer - 1] = 0xFFFFFFFFu;
      }
    }
    int rk[kPoolPer];  // position among the candidates of each of this lane's slots, or -1
#pragma unroll
    for (int k = 0; k < kPoolPer; ++k) rk[k] = -1;
#pragma unroll
    for (int j = 0; j < kPoolPer; ++j) {
      const int kj = static_cast<int>((pks >> (2 * j)) & 3u), aj = static_cast<int>((rks >> (4 * j)) & 15u);
#pragma unroll
      for (int k = 0; k < kPoolPer; ++k) rk[k] = (j < np && kj == k) ? aj : rk[k];
    }
    __syncwarp();
    // cos(c_a, c_b) for this lane's slots from row c_b (the block is
    // symmetric): one conflict-free 16-byte read per earlier candidate
    // (loads unconditional: every entry of s.pick is a valid slot, stale past r)
    unsigned int fail = 0;
#pragma unroll
    for (int c0 = 0; c0 < kPick; c0 += 4) {  // four reads in flight
      float4 c[4];
#pragma unroll
      for (int u = 0; u < 4; ++u) c[u] = *reinterpret_cast<const float4*>(&s.cp[s.pick[c0 + u]][kPoolPer * lane]);
#pragma unroll
      for (int u = 0; u < 4; ++u) {
        const int b2 = c0 + u;
        fail |= (b2 < rk[0] && c[u].x > pm[0]) ? 1u << rk[0] : 0u;
        fail |= (b2 < rk[1] && c[u].y > pm[1]) ? 1u << rk[1] : 0u;
        fail |= (b2 < rk[2] && c[u].z > pm[2]) ? 1u << rk[2] : 0u;
        fail |= (b2 < rk[3] && c[u].w > pm[3]) ? 1u << rk[3] : 0u;
      }
    }
    fail = __reduce_or_sync(0xFFFFFFFFu, fail);
    const int L = fail ? __ffs(fail) - 1 : r;  // bit 0 is never set
#pragma unroll
    for (int c0 = 0; c0 < kPick; c0 += 4) {
      float4 c[4];
#pragma unroll
      for (int u = 0; u < 4; ++u) c[u] = *reinterpret_cast<const float4*>(&s.cp[s.pick[c0 + u]][kPoolPer * lane]);
#pragma unroll
      for (int u = 0; u < 4; ++u) {
        const bool use = c0 + u < L;
        pm[0] = use ? fmaxf(pm[0], c[u].x) : pm[0]; pm[1] = use ? fmaxf(pm[1], c[u].y) : pm[1];
        pm[2] = use ? fmaxf(pm[2], c[u].z) : pm[2]; pm[3] = use ? fmaxf(pm[3], c[u].w) : pm[3];
      }
    }
#pragma unroll
    for (int k = 0; k < kPoolPer; ++k) {
      if (rk[k] >= 0 && rk[k] < L) {
        alive &= ~(1u << k);
        const int tok = s.ptok[kPoolPer * lane + k];
        s.list[npend + rk[k]] = tok;
        atomicOr(&s.keptbits[tok >> 5], 1u << (tok & 31));
      }
    }
    npend += L;
    t += L;
    __syncwarp();
  }
  if (lane == 0) {
    s.t = t;
    s.npend = npend;
  }
}

// kMode: kStagesAll runs stages 1-3 and writes idx; kStages12 runs stages 1-2
// and writes the kept set as bits (token t: bit t % 32 of word t / 32 of the
// image's row of kept12) so that it can run beside the cosine matrix; kStage3
// starts from those bits.
enum { kStagesAll = 0, kStages12 = 1, kStage3 = 2 };

template <int kMaxThreads, int kMode>
__global__ void __launch_bounds__(kMaxThreads, 1)
    select_stages_kernel(const float* __restrict__ scores, const float* __restrict__ A_cls,
                         const float* __restrict__ gram, int gp, int N, int J, int K, int Kq, int Ks,
                         int Kd, int32_t* __restrict__ idx, uint32_t* __restrict__ kept12) {
  pdl_wait();
  pdl_launch_dependents();
  extern __shared__ uint8_t smem_raw[];
  BlockScratch& s = *reinterpret_cast<BlockScratch*>(smem_raw);
  const int b = blockIdx.x;
  const int base = kPer * threadIdx.x;  // tokens of a group-0 thread (none for the other groups)
  const int tpg = ((N + kPer - 1) / kPer + 31) / 32 * 32, groups = blockDim.x / tpg;
  const bool g0 = threadIdx.x < tpg;
  bool kept[kPer];
#pragma unroll
  for (int e = 0; e < kPer; ++e) kept[e] = false;
  uint32_t key[kPer];
  const int words = (N + 31) / 32;

  if (kMode == kStage3) {
    if (g0) {
#pragma unroll
      for (int e = 0; e < kPer; ++e) {
        const int i = base + e;
        kept[e] = i < N && ((kept12[static_cast<size_t>(b) * words + (i >> 5)] >> (i & 31)) & 1u);
      }
    }
  } else if (g0) {
    // Stage 1: query relevance, one ranking per concept, quota floor(Kq/J) + (j < Kq % J).
    for (int j = 0; j < J && Kq > 0; ++j) {
      const int quota = Kq / J + (j < Kq % J ? 1 : 0);
      const float* sc = scores + (static_cast<size_t>(b) * J + j) * N;
#pragma unroll
      for (int e = 0; e < kPer; ++e) key[e] = (base + e < N) ? float_order_key(sc[base + e]) : 0u;
      block_take_top(key, kept, base, N, quota, tpg, s);
    }
    // Stage 2: visual saliency on the tokens not kept.
    if (Ks > 0) {
      const float* a = A_cls + static_cast<size_t>(b) * N;
#pragma unroll
      for (int e = 0; e < kPer; ++e) key[e] = (base + e < N) ? float_order_key(a[base + e]) : 0u;
      block_take_top(key, kept, base, N, Ks, tpg, s);
    }
  }
  if (kMode == kStages12) {
    for (int w = threadIdx.x; w < words; w += blockDim.x) s.keptbits[w] = 0u;
    __syncthreads();
    if (g0) {
#pragma unroll
      for (int e = 0; e < kPer; ++e)
        if (base + e < N && kept[e]) atomicOr(&s.keptbits[(base + e) >> 5], 1u << ((base + e) & 31));
    }
    __syncthreads();
    for (int w = threadIdx.x; w < words; w += blockDim.x) kept12[static_cast<size_t>(b) * words + w] = s.keptbits[w];
    return;
  }
  // Stage 3: greedy max-min diversity on the cosine matrix G of the image:
  // m_i = max over the kept set of cos(i, r) (-inf while it is empty); each
  // round keeps the free token with the smallest m (lower index on ties) and
  // m absorbs its cosines. Rounds run in phases on a pool of the smallest
  // free (m, token) pairs (pool_rounds); between phases the whole block
  // applies the pending rows and rebuilds the pool.
  if (Kd > 0) {
    const float* G = gram + static_cast<size_t>(b) * N * gp;
    for (int w = threadIdx.x; w < P4Q_MAX_TOKENS / 32; w += blockDim.x) s.keptbits[w] = 0u;
    if (threadIdx.x < kPick) s.pick[threadIdx.x] = 0;
    int nkept = 0, cnt = 0, pos = 0;
    if (g0) {
#pragma unroll
      for (int e = 0; e < kPer; ++e) cnt += (base + e < N && kept[e]) ? 1 : 0;
      pos = block_exclusive_scan(cnt, &nkept, tpg, s);
#pragma unroll
      for (int e = 0; e < kPer; ++e)
        if (base + e < N && kept[e]) s.list[pos++] = base + e;
      if (threadIdx.x == 0) {
        s.t = 0;
        s.npend = nkept;  // the kept set's rows come first
      }
    }
    __syncthreads();
    float m[kPer];
#pragma unroll
    for (int e = 0; e < kPer; ++e) m[e] = -INFINITY;
    for (int last = -1;;) {
      const int t = s.t;
#pragma unroll
      for (int e = 0; e < kPer; ++e)
        if (base + e < N && ((s.keptbits[(base + e) >> 5] >> ((base + e) & 31)) & 1u)) kept[e] = true;
      // every phase picks at least once (right after a rebuild the whole pool
      // is certain); the progress check only guards the loop
      if (t >= Kd || t == last) break;
      last = t;
      for (int i = threadIdx.x; i < N; i += blockDim.x) s.slotof[i] = -1;
      apply_rows(m, G, gp, N, s.npend, tpg, groups, s);
      int npool = 0;
      if (g0) {
        // pool: the q smallest free (m, token) pairs (radix select on inverted keys), in token order
        const int q = min(kPool, N - nkept - t);
        bool member[kPer];
#pragma unroll
        for (int e = 0; e < kPer; ++e) {
          member[e] = kept[e];
          key[e] = (base + e < N) ? ~float_order_key(m[e]) : 0u;
        }
        block_take_top(key, member, base, N, q, tpg, s);
        cnt = 0;
#pragma unroll
        for (int e = 0; e < kPer; ++e) cnt += (base + e < N && member[e] && !kept[e]) ? 1 : 0;
        pos = block_exclusive_scan(cnt, &npool, tpg, s);
#pragma unroll
        for (int e = 0; e < kPer; ++e) {
          if (base + e < N && member[e] && !kept[e]) {
            s.ptok[pos] = base + e;
            s.pm[pos] = m[e];
            s.slotof[base + e] = pos;
            ++pos;
          }
        }
        if (threadIdx.x == 0) s.npend = npool;  // rows of the pool tokens, for the cosine block
      }
      __syncthreads();
      npool = s.npend;
      // the pool's cosine block from whole rows of the pool tokens (coalesced):
      // each thread keeps the columns of its four tokens that are in the pool
      {
        const int g = threadIdx.x / tpg;
        const int tb = kPer * (threadIdx.x - g * tpg);
        int sl[kPer];
#pragma unroll
        for (int e = 0; e < kPer; ++e) sl[e] = (tb + e < N) ? s.slotof[tb + e] : -1;
        if (tb < N && (sl[0] >= 0 || sl[1] >= 0 || sl[2] >= 0 || sl[3] >= 0)) {
          for (int i0 = 8 * g; i0 < npool; i0 += 8 * groups) {
            float4 v[8];
#pragma unroll
            for (int u = 0; u < 8; ++u)
              v[u] = (i0 + u < npool) ? *reinterpret_cast<const float4*>(G + static_cast<size_t>(s.ptok[i0 + u]) * gp + tb)
                                      : make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
            for (int u = 0; u < 8; ++u) {
              if (i0 + u < npool) {
                float* row = s.cp[i0 + u];
                if (sl[0] >= 0) row[sl[0]] = v[u].x;
                if (sl[1] >= 0) row[sl[1]] = v[u].y;
                if (sl[2] >= 0) row[sl[2]] = v[u].z;
                if (sl[3] >= 0) row[sl[3]] = v[u].w;
              }
            }
          }
        }
      }
      __syncthreads();
      if (threadIdx.x < 32) pool_rounds(npool, Kd, s);
      __syncthreads();
    }
  }
  // Output: the kept set in ascending index order.
  if (g0) {
    int cnt = 0;
#pragma unroll
    for (int e = 0; e < kPer; ++e) cnt += (base + e < N && kept[e]) ? 1 : 0;
    int total;
    int pos = block_exclusive_scan(cnt, &total, tpg, s);
#pragma unroll
    for (int e = 0; e < kPer; ++e)
      if (base + e < N && kept[e] && pos < K) idx[static_cast<size_t>(b) * K + pos++] = base + e;
  }
}

size_t align256(size_t x) { return (x + 255) & ~static_cast<size_t>(255); }

// ---------------------------------------------------------------- Top-K replacement ratio
// App. A, Eq. 9: per sample, the Top-K sets of two score rows over the same N
// tokens (ties to the lower index, the selector's radix select) and the size
// of their intersection; rho = 1 - |T_ref & T_alt| / K. One CTA per sample,
// token i = kPer * threadIdx.x + e.
// Order key of a score with -0 and +0 equal (they tie, and the lower index wins).
__device__ __forceinline__ uint32_t score_key(float v) { return float_order_key(v == 0.0f ? 0.0f : v); }

struct TopkScratch {
  unsigned int hist[256];
  unsigned int wsum[32];
  int digit, above;
};

__global__ void __launch_bounds__(kSelThreads)
    topk_replacement_kernel(const float* __restrict__ s_ref, const float* __restrict__ s_alt, int N, int K,
                            int32_t* __restrict__ inter, float* __restrict__ rho) {
  pdl_wait();
  pdl_launch_dependents();
  __shared__ TopkScratch s;
  const int b = blockIdx.x, nt = blockDim.x, base = kPer * threadIdx.x;
  uint32_t key[kPer];
  bool in_ref[kPer], in_alt[kPer];
#pragma unroll
  for (int e = 0; e < kPer; ++e) {
    key[e] = base + e < N ? score_key(s_ref[static_cast<size_t>(b) * N + base + e]) : 0u;
    in_ref[e] = false;
    in_alt[e] = false;
  }
  block_take_top(key, in_ref, base, N, K, nt, s);
#pragma unroll
  for (int e = 0; e < kPer; ++e)
    key[e] = base + e < N ? score_key(s_alt[static_cast<size_t>(b) * N + base + e]) : 0u;
  block_take_top(key, in_alt, base, N, K, nt, s);
  int c = 0;
#pragma unroll
  for (int e = 0; e < kPer; ++e) c += (in_ref[e] && in_alt[e]) ? 1 : 0;
  int total;
  block_exclusive_scan(c, &total, nt, s);
  if (threadIdx.x == 0) {
    inter[b] = total;
    rho[b] = __fsub_rn(1.0f, __fdiv_rn(static_cast<float>(total), static_cast<float>(K)));
  }
}

}  // namespace

cudaError_t launch_topk_replacement(const float* s_ref, const float* s_alt, int B, int N, int K, int32_t* inter,
                                    float* rho, cudaStream_t stream) {
  if (B <= 0) return cudaSuccess;
  const int nt = ((N + kPer - 1) / kPer + 31) / 32 * 32;
  return launch_pdl(topk_replacement_kernel, dim3(B), dim3(nt), 0, stream, s_ref, s_alt, N, K, inter, rho);
}

size_t select_workspace_layout(int B, int N, int d, int J, SelectWorkspace* ws, void* base) {
  const size_t BN = static_cast<size_t>(B) * N, BJ = static_cast<size_t>(B) * J;
  size_t off = 0;
  auto take = [&](size_t bytes) {
    const size_t o = off;
    off += align256(bytes);
    return o;
  };
  const size_t o_vc = take(BN * (d / 2)), o_vs = take(BN * 4), o_vn = take(BN * 4);
  const size_t o_qc = take(BJ * (d / 2)), o_qs = take(BJ * 4), o_qn = take(BJ * 4);
  const int gp = (N + 3) & ~3;
  const size_t o_sc = take(BJ * N * 4), o_g = take(BN * gp * 4);
  const bool expanded = N >= kGramExpandedMin;
  const size_t o_vu = expanded ? take(BN * d) : 0, o_vsum = expanded ? take(BN * 4) : 0;
  const size_t o_k12 = take(static_cast<size_t>(B) * ((N + 31) / 32) * 4);
  if (ws && base) {
    uint8_t* p = static_cast<uint8_t*>(base);
    ws->vcodes = p + o_vc;
    ws->vscale = reinterpret_cast<float*>(p + o_vs);
    ws->vnorm = reinterpret_cast<int32_t*>(p + o_vn);
    ws->qcodes = p + o_qc;
    ws->qscale = reinterpret_cast<float*>(p + o_qs);
    ws->qnorm = reinterpret_cast<int32_t*>(p + o_qn);
    ws->scores = reinterpret_cast<float*>(p + o_sc);
    ws->gram = reinterpret_cast<float*>(p + o_g);
    ws->gram_pitch = gp;
    ws->vu = expanded ? p + o_vu : nullptr;
    ws->vsum = expanded ? reinterpret_cast<int32_t*>(p + o_vsum) : nullptr;
    ws->kept12 = reinterpret_cast<uint32_t*>(p + o_k12);
  }
  return off;
}

cudaError_t launch_query_scores(const SelectPlan& p, const SelectWorkspace& ws, cudaStream_t stream) {
  const size_t smem = static_cast<size_t>(p.J) * (p.d / 2);
  static size_t smem_set = 48u << 10;
  if (smem > smem_set) {
    cudaError_t e = cudaFuncSetAttribute(query_scores_kernel<P4Q_MAX_CONCEPTS>,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(smem));
    if (e != cudaSuccess) return e;
    smem_set = smem;
  }
  const dim3 grid((p.N + kScoreWarps - 1) / kScoreWarps, p.B);
  if (p.J <= 4)  // J * d / 2 <= 32 KB: no attribute needed
    return launch_pdl(query_scores_kernel<4>, grid, dim3(kScoreWarps * 32), smem, stream, ws.vcodes, ws.vnorm,
                      ws.qcodes, ws.qnorm, p.B, p.N, p.d, p.J, ws.scores);
  return launch_pdl(query_scores_kernel<P4Q_MAX_CONCEPTS>, grid, dim3(kScoreWarps * 32), smem, stream, ws.vcodes,
                    ws.vnorm, ws.qcodes, ws.qnorm, p.B, p.N, p.d, p.J, ws.scores);
}

namespace {

// The Gram buffer in place: int32 dot products in, the cosines out (same
// bits as the cosine epilogue of the GEMM). One warp per row at a time
// (grid-stride over rows), each lane two 16-byte chunks of four entries in
// flight; the IEEE division and square root make this instruction-bound.
__global__ void __launch_bounds__(256) gram_cos_kernel(float* __restrict__ gram, const int32_t* __restrict__ norm,
                                                       int N, int gp, int rows) {
  pdl_wait();
  pdl_launch_dependents();
  const int lane = threadIdx.x & 31;
  const int nwarps = gridDim.x * (blockDim.x >> 5);
  const int cpr = gp >> 2;  // chunks per row
  for (int row = blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5); row < rows; row += nwarps) {
    const int na = norm[row];
    const int32_t* nr = norm + (row / N) * N;  // norms of the image's tokens
    float* g = gram + static_cast<size_t>(row) * gp;
    for (int c0 = lane; c0 < cpr; c0 += 64) {
      int4 dv[2];
#pragma unroll
      for (int u = 0; u < 2; ++u) {
        const int c = c0 + 32 * u;
        dv[u] = c < cpr ? *reinterpret_cast<const int4*>(g + 4 * c) : make_int4(0, 0, 0, 0);
      }
#pragma unroll
      for (int u = 0; u < 2; ++u) {
        const int j = 4 * (c0 + 32 * u);
        if (j >= N) continue;
        float4 c;
        c.x = code_cosine(dv[u].x, na, nr[j]);
        c.y = (j + 1 < N) ? code_cosine(dv[u].y, na, nr[j + 1]) : 0.0f;
        c.z = (j + 2 < N) ? code_cosine(dv[u].z, na, nr[j + 2]) : 0.0f;
        c.w = (j + 3 < N) ? code_cosine(dv[u].w, na, nr[j + 3]) : 0.0f;
        *reinterpret_cast<float4*>(g + j) = c;
      }
    }
  }
}

}  // namespace

cudaError_t launch_gram_cos(const SelectPlan& p, const SelectWorkspace& ws, cudaStream_t stream) {
  const int rows = p.B * p.N;
  const int blocks = std::min((rows + 7) / 8, 8 * num_sms());
  return launch_pdl(gram_cos_kernel, dim3(blocks), dim3(256), 0, stream, ws.gram, ws.vnorm, p.N, ws.gram_pitch, rows);
}

cudaError_t launch_select_stages(const SelectPlan& p, const SelectWorkspace& ws, const float* A_cls, int32_t* idx,
                                 cudaStream_t stream, int mode) {
  static bool attr_set = false;
  const int smem = static_cast<int>(sizeof(BlockScratch));
  if (!attr_set) {
    const void* fns[] = {reinterpret_cast<const void*>(select_stages_kernel<kSelThreadsSmall, kStagesAll>),
                         reinterpret_cast<const void*>(select_stages_kernel<kSelThreadsSmall, kStages12>),
                         reinterpret_cast<const void*>(select_stages_kernel<kSelThreadsSmall, kStage3>),
                         reinterpret_cast<const void*>(select_stages_kernel<kSelThreadsMid, kStagesAll>),
                         reinterpret_cast<const void*>(select_stages_kernel<kSelThreads, kStagesAll>)};
    for (const void* f : fns) {
      cudaError_t e = cudaFuncSetAttribute(f, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
      if (e != cudaSuccess) return e;
    }
    attr_set = true;
  }
  // group 0: one thread per kPer tokens (idle threads would only add
  // instructions to every ranking); as many row groups as fit the block
  const int tpg = ((p.N + kPer - 1) / kPer + 31) / 32 * 32;
  if (tpg <= kSelThreadsSmall) {
    const dim3 block(tpg * (kSelThreadsSmall / tpg));
    if (mode == kStages12)
      return launch_pdl(select_stages_kernel<kSelThreadsSmall, kStages12>, dim3(p.B), dim3(tpg),
                        static_cast<size_t>(smem), stream, ws.scores, A_cls, ws.gram, ws.gram_pitch, p.N, p.J, p.K,
                        p.Kq, p.Ks, p.Kd, idx, ws.kept12);
    if (mode == kStage3)
      return launch_pdl(select_stages_kernel<kSelThreadsSmall, kStage3>, dim3(p.B), block, static_cast<size_t>(smem),
                        stream, ws.scores, A_cls, ws.gram, ws.gram_pitch, p.N, p.J, p.K, p.Kq, p.Ks, p.Kd, idx,
                        ws.kept12);
    return launch_pdl(select_stages_kernel<kSelThreadsSmall, kStagesAll>, dim3(p.B), block,
                      static_cast<size_t>(smem), stream, ws.scores, A_cls, ws.gram, ws.gram_pitch, p.N, p.J, p.K,
                      p.Kq, p.Ks, p.Kd, idx, ws.kept12);
  }
  if (mode != kStagesAll) return cudaErrorInvalidValue;  // split launches serve N <= 2048
  if (tpg <= kSelThreadsMid)
    return launch_pdl(select_stages_kernel<kSelThreadsMid, kStagesAll>, dim3(p.B), dim3(tpg * (kSelThreadsMid / tpg)),
                      static_cast<size_t>(smem), stream, ws.scores, A_cls, ws.gram, ws.gram_pitch, p.N, p.J, p.K,
                      p.Kq, p.Ks, p.Kd, idx, ws.kept12);
  return launch_pdl(select_stages_kernel<kSelThreads, kStagesAll>, dim3(p.B), dim3(tpg), static_cast<size_t>(smem),
                    stream, ws.scores, A_cls, ws.gram, ws.gram_pitch, p.N, p.J, p.K, p.Kq, p.Ks, p.Kd, idx,
                    ws.kept12);
}

bool select_split_applies(int N) { return ((N + kPer - 1) / kPer + 31) / 32 * 32 <= kSelThreadsSmall; }

}  // namespace p4q
