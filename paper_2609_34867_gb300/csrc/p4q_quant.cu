// Per-row symmetric 4-bit quantizer (App. A and App. B.3 of the paper:
// symmetric round-to-nearest, one scale per token or per output channel,
// group size -1, clip ratio 1.0), in fp32:
//   a = max_k |x_k|, s = a / 7 (rounded once), code_k = clamp(rne(x_k / s), -8, 7)
// with x_k / s rounded to fp32 before the round-half-even; a == 0 gives s = 0
// and zero codes. Codes are written packed, two per byte, the even index in
// the low nibble (two's complement).
//
// Kernels:
//   quant_rows_reg_kernel     dense rows of up to 16384 elements (a multiple
//                             of 256): each row held in the registers of one
//                             warp (up to 5120 elements) or of four, every
//                             load of a row in flight, the group's next row
//                             prefetched chunk by chunk as the current one is
//                             quantized. Activations, weights, the selector's
//                             concepts.
//   quant_rows_kernel         every other case (the fused gather of the
//                             pruned sequence through the kept indices with
//                             its fp16 copy, two row sets in one launch, other
//                             row lengths): rows stream through shared memory,
//                             a group of G warps owning a ring of S row
//                             buffers that its leader fills with bulk
//                             asynchronous copies (cp.async.bulk, one mbarrier
//                             per buffer); each row is read from shared memory
//                             twice (abs-max, then codes). Two persistent CTAs
//                             of 8 warps per SM.
//   select_token_quant_kernel the selector's tokens with the query dot
//                             products fused (register-resident, per image).
//   quant_rowmax_kernel       column blocks of a GEMM output whose row
//                             abs-max is known: one streaming pass.
// Optional outputs: the codes expanded one byte each (u = code + 8, the
// GEMM's operand form) with their row sums, and the squared code norm.
#include <cuda_fp16.h>

#include <algorithm>
#include <type_traits>

#include "p4q_device.cuh"
#include "p4q_internal.h"

namespace p4q {

// Device error word of the quantizer (bounded waits on the row buffers).
__device__ unsigned int g_quant_err;

namespace {

constexpr int kWarps = 8;
constexpr int kThreads = 32 * kWarps;
constexpr int kCtasPerSm = 2;
constexpr int kMaxStages = 16;
constexpr uint32_t kStageBudget = 100u * 1024u;    // shared memory for row buffers per CTA
constexpr uint32_t kInflightTarget = 48u * 1024u;  // bytes on their way per CTA (HBM latency x bandwidth share)
constexpr int kSmemMax = 110 * 1024;

// Codes of eight fp16 values (one 16-byte chunk).
//
// code = round_half_even(fl(x / s)). With inv = fl(1 / s) correctly rounded,
// fl(x / s) lies within 2^-23 (relative) of x * inv, so ip = fl(inv (1 +
// 2^-21)) and im = fl(inv (1 - 2^-21)) give products x * ip and x * im that
// enclose fl(x / s) (each is at least 2^-21 - 2^-23 away from x * inv). One
// fused multiply-add with the magic constant 1.5 * 2^23 rounds each exact
// product to the nearest integer (ties to even: the constant is even) and
// leaves its two's complement in the low mantissa bits. Rounding is
// monotone, so where the two agree their integer is the code of fl(x / s);
// a chunk where they differ for some value (a quotient within about 2^-21 of
// a .5 boundary) is recomputed with exact quotients fl(x / s). |x| <= max|x|
// bounds the codes to [-7, 7], so the clamp to [-8, 7] cannot bind. With
// NORM, squares of the codes are added to n2 (exact: sums below 2^24).
struct QRow {
  float s, ip, im;  // scale a / 7 and the two bracketing reciprocals (0 when a == 0)
};

__device__ __forceinline__ QRow quant_row(float a) {
  QRow r;
  r.s = __fdiv_rn(a, 7.0f);
  const float inv = (a != 0.0f) ? __frcp_rn(r.s) : 0.0f;
  r.ip = __fmul_rn(inv, 1.0f + 0x1p-21f);
  r.im = __fmul_rn(inv, 1.0f - 0x1p-21f);
  return r;
}

// Byte k of e holds the code of element 2k, byte k of o the code of element
// 2k + 1 (two's complement; the low nibble is the 4-bit code).
struct Codes8 {
  uint32_t e, o;
};

// packed: even-index codes in the low nibbles, odd-index codes in the high nibbles
__device__ __forceinline__ uint32_t packed4(Codes8 c) { return (c.e & 0x0F0F0F0Fu) | ((c.o << 4) & 0xF0F0F0F0u); }
// expanded, one byte per code u = v + 8: the four even-index codes, then the four odd-index codes
__device__ __forceinline__ uint32_t expanded_even(Codes8 c) { return (c.e & 0x0F0F0F0Fu) ^ 0x08080808u; }
__device__ __forceinline__ uint32_t expanded_odd(Codes8 c) { return (c.o & 0x0F0F0F0Fu) ^ 0x08080808u; }

template <bool NORM>
__device__ __forceinline__ Codes8 quant_chunk(const uint4 v, const QRow& q, float2& n2) {
  const float2 ip2 = make_float2(q.ip, q.ip), im2 = make_float2(q.im, q.im);
  const float2 mg = make_float2(12582912.0f, 12582912.0f);
  const uint32_t w[4] = {v.x, v.y, v.z, v.w};
  float2 f[4];
  uint32_t tb[8];
  uint32_t diff = 0;
#pragma unroll
  for (int k = 0; k < 4; ++k) {
    f[k] = __half22float2(*reinterpret_cast<const __half2*>(&w[k]));
    const float2 tp = __ffma2_rn(f[k], ip2, mg);
    const float2 tm = __ffma2_rn(f[k], im2, mg);
    tb[2 * k] = __float_as_uint(tp.x);
    tb[2 * k + 1] = __float_as_uint(tp.y);
    diff |= (tb[2 * k] ^ __float_as_uint(tm.x)) | (tb[2 * k + 1] ^ __float_as_uint(tm.y));
  }
  if (diff != 0) {
#pragma unroll
    for (int k = 0; k < 4; ++k) {
      tb[2 * k] = __float_as_uint(rintf(__fdiv_rn(f[k].x, q.s)) + 12582912.0f);
      tb[2 * k + 1] = __float_as_uint(rintf(__fdiv_rn(f[k].y, q.s)) + 12582912.0f);
    }
  }
  if (NORM) {
    const float2 nmg = make_float2(-12582912.0f, -12582912.0f);
#pragma unroll
    for (int k = 0; k < 4; ++k) {
      const float2 c = __fadd2_rn(make_float2(__uint_as_float(tb[2 * k]), __uint_as_float(tb[2 * k + 1])), nmg);
      n2 = __ffma2_rn(c, c, n2);
    }
  }
  Codes8 r;
  r.e = __byte_perm(__byte_perm(tb[0], tb[2], 0x0040), __byte_perm(tb[4], tb[6], 0x0040), 0x5410);
  r.o = __byte_perm(__byte_perm(tb[1], tb[3], 0x0040), __byte_perm(tb[5], tb[7], 0x0040), 0x5410);
  return r;
}

__device__ __forceinline__ const uint16_t* row_ptr(const RowSource& src, int row, int L) {
  if (src.X2 != nullptr && row >= src.split) return src.X2 + static_cast<size_t>(row - src.split) * L;
  if (src.idx == nullptr) return src.X + static_cast<size_t>(row) * (src.ldx > 0 ? src.ldx : L);
  const int per = src.K + src.T;
  const int b = row / per, r = row - b * per;
  if (r < src.K) return src.X + (static_cast<size_t>(b) * src.N + src.idx[b * src.K + r]) * L;
  return src.text + (static_cast<size_t>(b) * src.T + (r - src.K)) * L;
}

// Group g of CTA c takes rows first = c * kGroups + g, first + total, ...
// (total = gridDim.x * kGroups). Per row j of the group: wait for its buffer,
// abs-max pass, group reduction (named barrier when G > 1), quantize pass,
// release of the buffer to the leader, which refills it with row j + S.
// Waits are bounded; after a time-out the group keeps meeting its barriers
// but skips the work, and the leader waits (bounded) for the copies it has
// in flight before the CTA exits.
template <int G, bool NORM>
__global__ void __launch_bounds__(kThreads, kCtasPerSm)
    quant_rows_kernel(RowSource src, int rows, int L, RowSinks out1, RowSinks out2, int S, uint32_t stage_bytes) {
  constexpr int kGroups = kWarps / G;
  constexpr int kGroupThreads = 32 * G;
  extern __shared__ __align__(128) unsigned char smem[];
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int grp = warp / G;
  const int gt = (warp % G) * 32 + lane;  // thread index inside the group
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + static_cast<size_t>(kGroups) * S * stage_bytes);
  uint32_t* red = reinterpret_cast<uint32_t*>(bars + kGroups * kMaxStages);
  int* red_n = reinterpret_cast<int*>(red + kWarps);
  int* red_u = red_n + kWarps;
  int* aborts = red_u + kWarps;
  if (threadIdx.x < kGroups * S) mbar_init(&bars[threadIdx.x], 1);
  if (threadIdx.x < kGroups) aborts[threadIdx.x] = 0;
  fence_barrier_init();
  __syncthreads();
  pdl_wait();  // rows (and kept indices) come from the previous kernel
  pdl_launch_dependents();

  unsigned char* ring = smem + static_cast<size_t>(grp) * S * stage_bytes;
  uint64_t* full = bars + grp * S;
  volatile int* abort = aborts + grp;
  const int total = gridDim.x * kGroups;
  const int first = blockIdx.x * kGroups + grp;
  const int mine = rows > first ? (rows - first + total - 1) / total : 0;
  const uint32_t row_bytes = 2u * static_cast<uint32_t>(L);
  const int nch = L >> 3;  // 16-byte chunks per row
  const bool leader = gt == 0;

  int issued = 0;  // rows whose copy the leader has started
  if (leader) {
    for (; issued < S && issued < mine; ++issued) {
      mbar_arrive_expect_tx(&full[issued], row_bytes);
      bulk_load(ring + static_cast<size_t>(issued) * stage_bytes, row_ptr(src, first + issued * total, L), row_bytes,
                &full[issued]);
    }
  }
  bool failed = false;
  int consumed = 0;  // rows whose buffer this warp has seen complete
  for (int j = 0; j < mine; ++j) {
    const int st = j % S;
    const bool second = src.X2 != nullptr && first + j * total >= src.split;
    const RowSinks& out = second ? out2 : out1;
    const int row = second ? first + j * total - src.split : first + j * total;  // row of its sinks
    if (!failed) {
      failed = !mbar_wait_warp(&full[st], (j / S) & 1, abort, &g_quant_err);
      if (!failed) consumed = j + 1;
    }
    const uint4* v4 = reinterpret_cast<const uint4*>(ring + static_cast<size_t>(st) * stage_bytes);

    uint32_t m = 0;  // per-halfword max of |x| bit patterns (non-negative fp16 order as integers)
    if (!failed) {
#pragma unroll 4
      for (int c = gt; c < nch; c += kGroupThreads) {
        const uint4 v = v4[c];
        m = __vmaxu2(m, v.x & 0x7FFF7FFFu);
        m = __vmaxu2(m, v.y & 0x7FFF7FFFu);
        m = __vmaxu2(m, v.z & 0x7FFF7FFFu);
        m = __vmaxu2(m, v.w & 0x7FFF7FFFu);
      }
    }
    uint32_t mm = __reduce_max_sync(0xFFFFFFFFu, max(m & 0xFFFFu, m >> 16));
    if (G > 1) {
      if (lane == 0) red[warp] = mm;
      named_bar_sync(1 + grp, kGroupThreads);
#pragma unroll
      for (int w = 0; w < G; ++w) mm = max(mm, red[grp * G + w]);
    }
    const float a = __half2float(__ushort_as_half(static_cast<unsigned short>(mm)));
    const QRow qr = quant_row(a);

    float2 n2 = make_float2(0.0f, 0.0f);  // exact: sums of squared codes <= 49 * 16384 < 2^24
    uint32_t su = 0;                      // sum of the expanded codes u = v + 8 (expanded output)
    if (!failed) {
      uint32_t* q4 = out.codes ? reinterpret_cast<uint32_t*>(out.codes + static_cast<size_t>(row) * (L >> 1)) : nullptr;
      uint4* cp = out.copy ? reinterpret_cast<uint4*>(out.copy + static_cast<size_t>(row) * L) : nullptr;
      uint2* up = out.u ? reinterpret_cast<uint2*>(out.u + static_cast<size_t>(row) * L) : nullptr;
#pragma unroll 4
      for (int c = gt; c < nch; c += kGroupThreads) {
        const uint4 v = v4[c];
        const Codes8 cd = (a != 0.0f) ? quant_chunk<NORM>(v, qr, n2) : Codes8{0u, 0u};
        if (q4) q4[c] = packed4(cd);
        if (cp) cp[c] = v;
        if (up) {
          const uint32_t eu = expanded_even(cd), ou = expanded_odd(cd);
          up[c] = make_uint2(eu, ou);
          su = __dp4a(eu + ou, 0x01010101u, su);
        }
      }
    }
    int wn = 0, wu = 0;
    if (NORM) {
      wn = __reduce_add_sync(0xFFFFFFFFu, static_cast<int>(n2.x + n2.y));
      if (G > 1 && lane == 0) red_n[warp] = wn;
    }
    if (out.sum_u) {
      wu = static_cast<int>(__reduce_add_sync(0xFFFFFFFFu, su));
      if (G > 1 && lane == 0) red_u[warp] = wu;
    }
    // every warp of the group is done with buffer st (and has published red_n)
    if (G > 1)
      named_bar_sync(1 + grp, kGroupThreads);
    else
      __syncwarp();
    if (NORM && G > 1) {
      wn = 0;
#pragma unroll
      for (int w = 0; w < G; ++w) wn += red_n[grp * G + w];
    }
    if (out.sum_u && G > 1) {
      wu = 0;
#pragma unroll
      for (int w = 0; w < G; ++w) wu += red_u[grp * G + w];
    }
    if (leader) {
      if (!failed) {
        out.scale[row] = (a != 0.0f) ? qr.s : 0.0f;
        if (NORM) out.norm2[row] = wn;
        if (out.sum_u) out.sum_u[row] = wu;
        if (issued < mine) {
          mbar_arrive_expect_tx(&full[st], row_bytes);
          bulk_load(ring + static_cast<size_t>(st) * stage_bytes, row_ptr(src, first + issued * total, L), row_bytes,
                    &full[st]);
          ++issued;
        }
      }
    }
  }
  if (leader && failed) {
    // leave no copy in flight into this CTA's shared memory
    int fresh = 0;
    for (int j = consumed; j < issued; ++j)
      mbar_wait(&full[j % S], (j / S) & 1, reinterpret_cast<volatile int*>(&fresh), &g_quant_err, 100000000ull);
  }
}

struct Plan {
  int G, S;
  uint32_t stage_bytes;
};

// Smallest group size whose ring keeps kInflightTarget bytes on their way
// (groups x (S - 1) buffers), else the one that keeps the most.
Plan plan_for(int L) {
  const uint32_t sb = (2u * static_cast<uint32_t>(L) + 127u) & ~127u;
  Plan best{kWarps, 2, sb};
  uint64_t best_inflight = 0;
  for (int G = 1; G <= kWarps; G *= 2) {
    const int groups = kWarps / G;
    const int S = std::min<int>(kMaxStages, static_cast<int>(kStageBudget / (groups * sb)));
    if (S < 2) continue;
    const uint64_t inflight = static_cast<uint64_t>(groups) * (S - 1) * sb;
    if (inflight >= kInflightTarget) return Plan{G, S, sb};
    if (inflight > best_inflight) {
      best = Plan{G, S, sb};
      best_inflight = inflight;
    }
  }
  return best;
}

int sm_count() {
  static int n = 0;
  if (n == 0) {
    int dev = 0;
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev);
    if (n <= 0) n = 1;
  }
  return n;
}

template <int G, bool NORM>
cudaError_t launch_g(const RowSource& src, int rows, int L, const RowSinks& out, const RowSinks& out2, const Plan& p,
                     cudaStream_t stream) {
  static bool attr_set = false;
  if (!attr_set) {
    cudaError_t e = cudaFuncSetAttribute(quant_rows_kernel<G, NORM>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         kSmemMax);
    if (e != cudaSuccess) return e;
    attr_set = true;
  }
  constexpr int kGroups = kWarps / G;
  const size_t smem = static_cast<size_t>(kGroups) * p.S * p.stage_bytes + kGroups * kMaxStages * 8 +
                      3 * kWarps * 4 + kGroups * 4;
  const int need = (rows + kGroups - 1) / kGroups;
  const int grid = std::min(need, kCtasPerSm * sm_count());
  return launch_pdl(quant_rows_kernel<G, NORM>, dim3(grid), dim3(kThreads), smem, stream, src, rows, L, out, out2,
                    p.S, p.stage_bytes);
}

template <bool NORM>
cudaError_t launch_norm(const RowSource& src, int rows, int L, const RowSinks& out, const RowSinks& out2,
                        cudaStream_t stream) {
  const Plan p = plan_for(L);
  switch (p.G) {
    case 1: return launch_g<1, NORM>(src, rows, L, out, out2, p, stream);
    case 2: return launch_g<2, NORM>(src, rows, L, out, out2, p, stream);
    case 4: return launch_g<4, NORM>(src, rows, L, out, out2, p, stream);
    default: return launch_g<8, NORM>(src, rows, L, out, out2, p, stream);
  }
}

// ---------------------------------------------------------------- selector token pass
// The selector's fake-quantized tokens (the quantizer above with the squared
// code norm and the expanded codes) with the Eq. 4 query dot products fused:
// one warp per token row, the row held in registers (CH 16-byte chunks per
// lane, all loads of a row in flight at once), the abs-max a warp reduction,
// no shared-memory pass and no block barrier. CTA (x, b) takes rows of image
// b only, so the image's J concept rows (expanded codes, written by the
// concept pass before this launch) sit in shared memory and each chunk's
// bytes u are multiplied into them by dp4a as they are produced: the exact
// code dot product with concept j is sum u u_j - 8 sum u - 8 sum u_j + 64 L.
// Rolling prefetch: as soon as a chunk is quantized its registers take the
// same chunk of the warp's next row, so the next row's loads are in flight
// during the rest of this row's work without more registers.
template <int CH, int JMAX>
__global__ void __launch_bounds__(256, 2)
    select_token_quant_kernel(const uint16_t* __restrict__ V, int N, int L, int J, const uint8_t* __restrict__ qu,
                              const int32_t* __restrict__ qsum, RowSinks out, float* __restrict__ qdots, int qp) {
  extern __shared__ __align__(16) uint8_t cq[];  // [J, L] the image's concept codes, expanded
  const int b = blockIdx.y, lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  pdl_wait();  // the concept codes come from the previous launch
  pdl_launch_dependents();
  if (JMAX > 0) {
    const uint4* src = reinterpret_cast<const uint4*>(qu + static_cast<size_t>(b) * J * L);
    for (int i = threadIdx.x; i < J * L / 16; i += blockDim.x) reinterpret_cast<uint4*>(cq)[i] = src[i];
    __syncthreads();
  }
  const int nch = L >> 3;
  const int wpi = gridDim.x * (blockDim.x >> 5);  // warps per image
  const int r_first = blockIdx.x * (blockDim.x >> 5) + warp;
  uint4 v[CH];
  if (r_first < N) {
    const uint4* x = reinterpret_cast<const uint4*>(V + (static_cast<size_t>(b) * N + r_first) * L);
#pragma unroll
    for (int i = 0; i < CH; ++i) {
      const int c = lane + 32 * i;
      v[i] = (c < nch) ? ldg_stream16(x + c) : make_uint4(0u, 0u, 0u, 0u);
    }
  }
  for (int r = r_first; r < N; r += wpi) {
    const size_t row = static_cast<size_t>(b) * N + r;
    const bool more = r + wpi < N;
    const uint4* xn = reinterpret_cast<const uint4*>(V + (row + (more ? wpi : 0)) * L);  // the warp's next row
    uint32_t m = 0;  // per-halfword max of |x| bit patterns
#pragma unroll
    for (int i = 0; i < CH; ++i) {
      m = __vmaxu2(m, v[i].x & 0x7FFF7FFFu);
      m = __vmaxu2(m, v[i].y & 0x7FFF7FFFu);
      m = __vmaxu2(m, v[i].z & 0x7FFF7FFFu);
      m = __vmaxu2(m, v[i].w & 0x7FFF7FFFu);
    }
    const uint32_t mm = __reduce_max_sync(0xFFFFFFFFu, max(m & 0xFFFFu, m >> 16));
    const float a = __half2float(__ushort_as_half(static_cast<unsigned short>(mm)));
    const QRow qr = quant_row(a);
    float2 n2 = make_float2(0.0f, 0.0f);  // unused: the norm comes from the expanded codes
    uint32_t su = 0, uu = 0;              // sums of u and of u^2
    uint32_t dq[JMAX > 0 ? JMAX : 1];
#pragma unroll
    for (int j = 0; j < (JMAX > 0 ? JMAX : 1); ++j) dq[j] = 0;
    uint2* up = reinterpret_cast<uint2*>(out.u + row * L);
#pragma unroll
    for (int i = 0; i < CH; ++i) {
      const int c = lane + 32 * i;
      if (c < nch) {
        const Codes8 cd = (a != 0.0f) ? quant_chunk<false>(v[i], qr, n2) : Codes8{0u, 0u};
        if (more) v[i] = ldg_stream16(xn + c);
        const uint32_t eu = expanded_even(cd), ou = expanded_odd(cd);
        up[c] = make_uint2(eu, ou);
        su = __dp4a(eu + ou, 0x01010101u, su);
        uu = __dp4a(eu, eu, __dp4a(ou, ou, uu));
#pragma unroll
        for (int j = 0; j < JMAX; ++j) {
          if (j < J) {
            const uint2 w = *reinterpret_cast<const uint2*>(cq + static_cast<size_t>(j) * L + 8 * c);
            dq[j] = __dp4a(eu, w.x, __dp4a(ou, w.y, dq[j]));
          }
        }
      }
    }
    const int wu = static_cast<int>(__reduce_add_sync(0xFFFFFFFFu, su));
    // sum of squared codes (u - 8)^2 over the row's L codes, exactly
    const int wn = static_cast<int>(__reduce_add_sync(0xFFFFFFFFu, uu)) - 16 * wu + 64 * L;
#pragma unroll
    for (int j = 0; j < JMAX; ++j) {
      if (j < J) {
        const int p = static_cast<int>(__reduce_add_sync(0xFFFFFFFFu, dq[j]));
        if (lane == j) {
          // exact (|dot| <= 49 L < 2^24), so the float holds it exactly
          const int dot = p - 8 * wu - 8 * qsum[b * J + j] + 64 * L;
          qdots[row * qp + j] = static_cast<float>(dot);
        }
      }
    }
    if (lane == 0) {
      out.scale[row] = (a != 0.0f) ? qr.s : 0.0f;
      out.norm2[row] = wn;
      out.sum_u[row] = wu;
    }
  }
}

template <int CH, int JMAX>
cudaError_t launch_token_quant(const uint16_t* V, int B, int N, int L, int J, const uint8_t* qu, const int32_t* qsum,
                               const RowSinks& out, float* qdots, int qp, cudaStream_t stream) {
  const size_t smem = static_cast<size_t>(J) * L;
  static bool attr_set = false;
  if (!attr_set) {
    cudaError_t e = cudaFuncSetAttribute(select_token_quant_kernel<CH, JMAX>,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize, 100 * 1024);
    if (e != cudaSuccess) return e;
    attr_set = true;
  }
  // at most two CTAs of 8 warps per SM over the whole batch (one wave: rows are dealt out per CTA in
  // advance, so a second wave would double the time), never more warps than an image has rows
  const int per_image = std::max(1, std::min((N + 7) / 8, 2 * sm_count() / B));
  return launch_pdl(select_token_quant_kernel<CH, JMAX>, dim3(per_image, B), dim3(256), smem, stream, V, N, L, J, qu,
                    qsum, out, qdots, qp);
}

// ---------------------------------------------------------------- known row abs-max
// Up to two column blocks of Y quantized per row with the abs-max already
// known (the GEMM's row-max epilogue): no abs-max pass, no reduction before
// the codes, so G warps stream a block row in 256-element steps (one 16-byte
// chunk per lane, steps interleaved over the G warps, kRmUnroll in flight per
// warp) and only the row sum of the expanded codes is reduced at the end. The
// pass is issue-bound (about 14 instructions per code at a quarter of the
// warp slots), so a few thousand rows (the short sequences) take G = 2 or 4
// warps per row to fill the GPU; G = 1 otherwise. Same arithmetic as
// quant_rows_kernel (s = a / 7, quant_chunk), so the same codes and scales.
struct RowmaxArgs {
  const uint16_t* Y;
  int ldy, M, nblk;
  RowmaxBlock b[2];
  const uint32_t* rowmax;
};

constexpr int kRmUnroll = 4;  // 256-element steps in flight per warp

template <int G>
__global__ void __launch_bounds__(256, 4) quant_rowmax_kernel(RowmaxArgs a) {
  __shared__ uint32_t red[2][8];  // per warp: its part of the row sum (two buffers: one barrier per row)
  pdl_wait();  // Y and its row maxima come from the previous kernel
  pdl_launch_dependents();
  constexpr int kRows = 8 / G;  // rows in flight per CTA
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int grp = warp / G, seg = warp % G;
  const int tasks = a.nblk * a.M;
  int par = 0;
  for (int t = blockIdx.x * kRows + grp; t < tasks; t += gridDim.x * kRows, par ^= 1) {  // uniform across the group
    const int bi = t / a.M, m = t - bi * a.M;
    const bool b1 = bi != 0;  // field by field: no dynamic index into the parameter array
    RowmaxBlock B;
    B.col0 = b1 ? a.b[1].col0 : a.b[0].col0;
    B.L = b1 ? a.b[1].L : a.b[0].L;
    B.codes = b1 ? a.b[1].codes : a.b[0].codes;
    B.scale = b1 ? a.b[1].scale : a.b[0].scale;
    B.u = b1 ? a.b[1].u : a.b[0].u;
    B.sum_u = b1 ? a.b[1].sum_u : a.b[0].sum_u;
    const float amax = __half2float(__ushort_as_half(static_cast<unsigned short>(a.rowmax[t])));
    const QRow qr = quant_row(amax);
    const uint4* x = reinterpret_cast<const uint4*>(a.Y + static_cast<size_t>(m) * a.ldy + B.col0);
    uint32_t* q4 = B.codes ? reinterpret_cast<uint32_t*>(B.codes + static_cast<size_t>(m) * (B.L >> 1)) : nullptr;
    uint2* up = reinterpret_cast<uint2*>(B.u + static_cast<size_t>(m) * B.L);
    const int steps = B.L >> 8;  // 256 elements per warp step
    float2 n2 = make_float2(0.0f, 0.0f);
    uint32_t su = 0;
    for (int j0 = seg; j0 < steps; j0 += kRmUnroll * G) {
      uint4 v[kRmUnroll];
#pragma unroll
      for (int k = 0; k < kRmUnroll; ++k) {
        const int j = j0 + k * G;
        v[k] = (j < steps) ? ldg_stream16(x + j * 32 + lane) : make_uint4(0u, 0u, 0u, 0u);
      }
#pragma unroll
      for (int k = 0; k < kRmUnroll; ++k) {
        const int j = j0 + k * G;
        if (j < steps) {
          const int c = j * 32 + lane;
          const Codes8 cd = (amax != 0.0f) ? quant_chunk<false>(v[k], qr, n2) : Codes8{0u, 0u};
          if (q4) q4[c] = packed4(cd);
          const uint32_t eu = expanded_even(cd), ou = expanded_odd(cd);
          up[c] = make_uint2(eu, ou);
          su = __dp4a(eu + ou, 0x01010101u, su);
        }
      }
    }
    uint32_t wu = __reduce_add_sync(0xFFFFFFFFu, su);
    if (G > 1) {
      if (lane == 0) red[par][warp] = wu;
      named_bar_sync(1 + grp, 32 * G);
      wu = 0;
#pragma unroll
      for (int i = 0; i < G; ++i) wu += red[par][grp * G + i];
    }
    if (seg == 0 && lane == 0) {
      B.scale[m] = (amax != 0.0f) ? qr.s : 0.0f;
      B.sum_u[m] = static_cast<int>(wu);
    }
  }
}

// ---------------------------------------------------------------- dense rows in registers
// Dense rows of L <= kRegRowMax elements (L % 256 == 0): a group of G warps
// per row, the row in registers (CH 16-byte chunks per thread, all loads of
// a row in flight), abs-max by warp reductions (and, for G > 1, a named
// barrier of the group), and the rolling prefetch of the group's next row
// (as in the selector's token pass). Same arithmetic as quant_rows_kernel;
// NORM takes the squared code norm from the expanded codes by dp4a.
constexpr int kRegRowMax = 16384;
constexpr int kRegMinRows = 2048;

template <int CH, int G, bool NORM>
__global__ void __launch_bounds__(256, 2)
    quant_rows_reg_kernel(const uint16_t* __restrict__ X, long long ldx, int rows, int L, RowSinks out) {
  __shared__ uint32_t red[8][3];  // per warp: abs-max, sum of u, sum of u^2 (G > 1)
  pdl_wait();  // rows come from the previous kernel
  pdl_launch_dependents();
  constexpr int kGroups = 8 / G;
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int grp = warp / G, gt = (warp % G) * 32 + lane;  // thread index inside the group
  const int nch = L >> 3;
  const int groups = gridDim.x * kGroups;
  const int r_first = blockIdx.x * kGroups + grp;
  uint4 v[CH];
  if (r_first < rows) {
    const uint4* x = reinterpret_cast<const uint4*>(X + static_cast<size_t>(r_first) * ldx);
#pragma unroll
    for (int i = 0; i < CH; ++i) {
      const int c = gt + 32 * G * i;
      v[i] = (c < nch) ? ldg_stream16(x + c) : make_uint4(0u, 0u, 0u, 0u);
    }
  }
  for (int r = r_first; r < rows; r += groups) {  // uniform across the group
    const bool more = r + groups < rows;
    const uint4* xn = reinterpret_cast<const uint4*>(X + static_cast<size_t>(more ? r + groups : r) * ldx);
    uint32_t m = 0;
#pragma unroll
    for (int i = 0; i < CH; ++i) {
      m = __vmaxu2(m, v[i].x & 0x7FFF7FFFu);
      m = __vmaxu2(m, v[i].y & 0x7FFF7FFFu);
      m = __vmaxu2(m, v[i].z & 0x7FFF7FFFu);
      m = __vmaxu2(m, v[i].w & 0x7FFF7FFFu);
    }
    uint32_t mm = __reduce_max_sync(0xFFFFFFFFu, max(m & 0xFFFFu, m >> 16));
    if (G > 1) {
      if (lane == 0) red[warp][0] = mm;
      named_bar_sync(1 + grp, 32 * G);
#pragma unroll
      for (int w = 0; w < G; ++w) mm = max(mm, red[grp * G + w][0]);
    }
    const float a = __half2float(__ushort_as_half(static_cast<unsigned short>(mm)));
    const QRow qr = quant_row(a);
    float2 n2 = make_float2(0.0f, 0.0f);  // unused: NORM comes from the expanded codes
    uint32_t su = 0, uu = 0;
    uint32_t* q4 = out.codes ? reinterpret_cast<uint32_t*>(out.codes + static_cast<size_t>(r) * (L >> 1)) : nullptr;
    uint2* up = out.u ? reinterpret_cast<uint2*>(out.u + static_cast<size_t>(r) * L) : nullptr;
#pragma unroll
    for (int i = 0; i < CH; ++i) {
      const int c = gt + 32 * G * i;
      if (c < nch) {
        const Codes8 cd = (a != 0.0f) ? quant_chunk<false>(v[i], qr, n2) : Codes8{0u, 0u};
        if (more) v[i] = ldg_stream16(xn + c);
        if (q4) q4[c] = packed4(cd);
        const uint32_t eu = expanded_even(cd), ou = expanded_odd(cd);
        if (up) up[c] = make_uint2(eu, ou);
        su = __dp4a(eu + ou, 0x01010101u, su);
        if (NORM) uu = __dp4a(eu, eu, __dp4a(ou, ou, uu));
      }
    }
    int wu = static_cast<int>(__reduce_add_sync(0xFFFFFFFFu, su));
    int wuu = NORM ? static_cast<int>(__reduce_add_sync(0xFFFFFFFFu, uu)) : 0;
    if (G > 1) {
      if (lane == 0) {
        red[warp][1] = static_cast<uint32_t>(wu);
        red[warp][2] = static_cast<uint32_t>(wuu);
      }
      named_bar_sync(1 + grp, 32 * G);
      wu = wuu = 0;
#pragma unroll
      for (int w = 0; w < G; ++w) {
        wu += static_cast<int>(red[grp * G + w][1]);
        wuu += static_cast<int>(red[grp * G + w][2]);
      }
    }
    if (gt == 0) {
      out.scale[r] = (a != 0.0f) ? qr.s : 0.0f;
      if (NORM) out.norm2[r] = wuu - 16 * wu + 64 * L;
      if (out.sum_u) out.sum_u[r] = wu;
    }
    if (G > 1) named_bar_sync(1 + grp, 32 * G);  // the group's reductions are read before the next row writes them
  }
}

template <int CH, int G, bool NORM>
cudaError_t launch_reg(const RowSource& src, int rows, int L, const RowSinks& out, cudaStream_t stream) {
  const long long ldx = src.ldx > 0 ? src.ldx : L;
  const int groups = 8 / G;
  const int blocks = std::max(1, std::min((rows + groups - 1) / groups, 2 * sm_count()));  // one wave
  return launch_pdl(quant_rows_reg_kernel<CH, G, NORM>, dim3(blocks), dim3(256), 0, stream, src.X, ldx, rows, L,
                    out);
}

// One warp per row up to 5120 elements (at most 20 chunks per lane), else a
// group of 4 warps (at most 16 chunks per thread: 16384 elements).
template <bool NORM>
cudaError_t launch_reg_norm(const RowSource& src, int rows, int L, const RowSinks& out, cudaStream_t stream) {
  const int ch = L / 256;
  if (ch <= 4) return launch_reg<4, 1, NORM>(src, rows, L, out, stream);
  if (ch <= 8) return launch_reg<8, 1, NORM>(src, rows, L, out, stream);
  if (ch <= 12) return launch_reg<12, 1, NORM>(src, rows, L, out, stream);
  if (ch <= 16) return launch_reg<16, 1, NORM>(src, rows, L, out, stream);
  if (ch <= 20) return launch_reg<20, 1, NORM>(src, rows, L, out, stream);
  const int ch4 = (ch + 3) / 4;
  if (ch4 <= 12) return launch_reg<12, 4, NORM>(src, rows, L, out, stream);
  return launch_reg<16, 4, NORM>(src, rows, L, out, stream);
}

}  // namespace

cudaError_t launch_quant_rowmax(const uint16_t* Y, int ldy, int M, int nblk, const RowmaxBlock* blk,
                                const uint32_t* rowmax, cudaStream_t stream) {
  if (M <= 0) return cudaSuccess;
  if (nblk < 1 || nblk > 2 || !Y || !rowmax) return cudaErrorInvalidValue;
  RowmaxArgs a;
  a.Y = Y;
  a.ldy = ldy;
  a.M = M;
  a.nblk = nblk;
  a.rowmax = rowmax;
  for (int i = 0; i < nblk; ++i) {
    if (blk[i].L <= 0 || blk[i].L % 256 != 0 || !blk[i].scale || !blk[i].u || !blk[i].sum_u)
      return cudaErrorInvalidValue;
    a.b[i] = blk[i];
  }
  // warps per row: as many as fill the resident warp slots (32 per SM at the
  // kernel's registers), at most one per 256-element step of the shorter block
  const int tasks = nblk * M;
  const int steps = std::min(a.b[0].L, a.b[nblk - 1].L) >> 8;
  const long long slots = 32LL * sm_count();
  const int G = (4LL * tasks <= slots && steps >= 4) ? 4 : (2LL * tasks <= slots && steps >= 2) ? 2 : 1;
  const int rows_per_cta = 8 / G;
  const int blocks = std::max(1, std::min((tasks + rows_per_cta - 1) / rows_per_cta, 8 * sm_count()));
  if (G == 4) return launch_pdl(quant_rowmax_kernel<4>, dim3(blocks), dim3(256), 0, stream, a);
  if (G == 2) return launch_pdl(quant_rowmax_kernel<2>, dim3(blocks), dim3(256), 0, stream, a);
  return launch_pdl(quant_rowmax_kernel<1>, dim3(blocks), dim3(256), 0, stream, a);
}

bool select_token_quant_applies(int d, int J) {
  return d % 256 == 0 && d <= kTokenQuantMaxRow && static_cast<size_t>(J) * d <= 96u * 1024u;
}

cudaError_t launch_select_token_quant(const uint16_t* V, int B, int N, int d, int J, const uint8_t* qu,
                                      const int32_t* qsum, const RowSinks& out, float* qdots, int qp,
                                      cudaStream_t stream) {
  if (!select_token_quant_applies(d, J) || !out.u || !out.sum_u || !out.norm2 || !out.scale) return cudaErrorInvalidValue;
  if (J > 0 && (!qu || !qsum || !qdots)) return cudaErrorInvalidValue;
  const int ch = d / 256;
  auto go = [&](auto ch_tag) -> cudaError_t {
    constexpr int C = decltype(ch_tag)::value;
    if (J == 0) return launch_token_quant<C, 0>(V, B, N, d, J, qu, qsum, out, qdots, qp, stream);
    if (J <= 4) return launch_token_quant<C, 4>(V, B, N, d, J, qu, qsum, out, qdots, qp, stream);
    return launch_token_quant<C, 16>(V, B, N, d, J, qu, qsum, out, qdots, qp, stream);
  };
  if (ch <= 4) return go(std::integral_constant<int, 4>());
  if (ch <= 8) return go(std::integral_constant<int, 8>());
  if (ch <= 12) return go(std::integral_constant<int, 12>());
  if (ch <= 16) return go(std::integral_constant<int, 16>());
  return go(std::integral_constant<int, 20>());
}


cudaError_t launch_quant_rows(const RowSource& src, int rows, int L, const RowSinks& out,
                              cudaStream_t stream, const RowSinks* out2) {
  if (rows <= 0) return cudaSuccess;
  if (src.X2 != nullptr && (out2 == nullptr || out2->codes == nullptr || out2->scale == nullptr || src.idx != nullptr ||
                            src.ldx != 0 || (out.norm2 == nullptr) != (out2->norm2 == nullptr)))
    return cudaErrorInvalidValue;
  // packed codes may be left out when the expanded ones are written
  if (out.scale == nullptr || (out.codes == nullptr && out.u == nullptr)) return cudaErrorInvalidValue;
  const RowSinks& o2 = out2 ? *out2 : out;
  // dense rows of at most kRegRowMax elements, at least a wave of them: the
  // register-resident kernel (a few rows, e.g. the selector's concepts, run
  // faster in the chain on the ring kernel: measured 85 against 95 us per
  // 8 x 576 selector call)
  if (rows >= kRegMinRows && src.X2 == nullptr && src.idx == nullptr && out.copy == nullptr && L % 256 == 0 &&
      L <= kRegRowMax && (out.u == nullptr) == (out.sum_u == nullptr))
    return out.norm2 ? launch_reg_norm<true>(src, rows, L, out, stream) : launch_reg_norm<false>(src, rows, L, out, stream);
  return out.norm2 ? launch_norm<true>(src, rows, L, out, o2, stream)
                   : launch_norm<false>(src, rows, L, out, o2, stream);
}

unsigned int quant_read_and_clear_error() {
  unsigned int v = 0, z = 0;
  cudaMemcpyFromSymbol(&v, g_quant_err, sizeof(v));
  cudaMemcpyToSymbol(g_quant_err, &z, sizeof(z));
  return v;
}

}  // namespace p4q
