// Block-level ranking helpers of the selector kernels (Sec. 3.2, Eq. 4:
// every stage keeps the best-ranked tokens, ties to the lower token index).
// Token i of an image is held by thread i / kPer of the block's first nt
// threads (element i % kPer); the other threads of the block do not take part.
#pragma once

#include <cstdint>

#include "p4q_device.cuh"

namespace p4q {

constexpr int kPer = 4;  // tokens per ranking thread: token i = kPer * threadIdx.x + e

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

}  // namespace p4q
