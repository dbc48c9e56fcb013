// Block objective of the pruning-aware calibration (Sec. 3.3, Eq. 5): for
// each calibration sample n with m_n rows of the block's output (rows
// off[n] .. off[n+1]-1 of the W4A4 output Yq and of the full-precision
// output Yf, d columns each)
//   e_n = ||Yq_n - Yf_n||_F^2 / (m_n d),   L = (1/B) sum_n e_n.
//
// The sample offsets come from the host (validated there) inside the launch
// parameters. Two launches, deterministic: grid (C, B) CTAs each sum the squared
// differences of the rows c, c + C, ... of sample n (fp16 pairs widened to
// fp32, four 16-byte chunk pairs in flight per thread, squares summed in fp32
// per thread over a few hundred values, the
// threads' sums combined in fp64 in a fixed order) into a partial; one CTA
// then adds each sample's C partials in order, divides, and averages over the
// samples in order.
#include <cuda_fp16.h>

#include "p4q.h"
#include "p4q_device.cuh"
#include "p4q_internal.h"

namespace p4q {
namespace {

constexpr int kMseThreads = 256;
constexpr int kMseUnroll = 4;  // 16-byte chunk pairs in flight per thread

struct MseParams {
  long long ldq, ldf;
  int B, d;
  int off[kMseMaxSamples + 1];
};

__device__ __forceinline__ double block_sum_f64(double v, double* red) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xFFFFFFFFu, v, o);
  if (lane == 0) red[warp] = v;
  __syncthreads();
  double t = 0.0;
  for (int w = 0; w < static_cast<int>(blockDim.x >> 5); ++w) t += red[w];
  return t;
}

__global__ void __launch_bounds__(kMseThreads)
    mse_partial_kernel(const __half* __restrict__ Yq, const __half* __restrict__ Yf, const MseParams p,
                       double* __restrict__ partial) {
  pdl_wait();
  pdl_launch_dependents();
  __shared__ double red[kMseThreads / 32];
  const int c = blockIdx.x, C = gridDim.x, n = blockIdx.y;
  const int r0 = p.off[n], r1 = p.off[n + 1];
  const int nch = p.d >> 3;
  // the (row, chunk) pairs of this CTA, kMseUnroll of them in flight per thread
  const int nrows = r1 > r0 + c ? (r1 - r0 - c + C - 1) / C : 0;
  const int items = nrows * nch;
  float acc = 0.0f;
  for (int i0 = threadIdx.x; i0 < items; i0 += kMseThreads * kMseUnroll) {
    uint4 a[kMseUnroll], f[kMseUnroll];
#pragma unroll
    for (int u = 0; u < kMseUnroll; ++u) {
      const int i = i0 + u * kMseThreads;
      if (i < items) {
        const int rr = i / nch, k = i - rr * nch;
        const size_t r = static_cast<size_t>(r0 + c + rr * C);
        a[u] = __ldg(reinterpret_cast<const uint4*>(Yq + r * p.ldq) + k);
        f[u] = __ldg(reinterpret_cast<const uint4*>(Yf + r * p.ldf) + k);
      } else {
        a[u] = make_uint4(0u, 0u, 0u, 0u);
        f[u] = a[u];
      }
    }
#pragma unroll
    for (int u = 0; u < kMseUnroll; ++u) {
      const uint32_t aw[4] = {a[u].x, a[u].y, a[u].z, a[u].w}, fw[4] = {f[u].x, f[u].y, f[u].z, f[u].w};
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        const float2 av = __half22float2(*reinterpret_cast<const __half2*>(&aw[e]));
        const float2 fv = __half22float2(*reinterpret_cast<const __half2*>(&fw[e]));
        const float d0 = av.x - fv.x, d1 = av.y - fv.y;
        acc = fmaf(d0, d0, acc);
        acc = fmaf(d1, d1, acc);
      }
    }
  }
  const double t = block_sum_f64(static_cast<double>(acc), red);
  if (threadIdx.x == 0) partial[static_cast<size_t>(n) * C + c] = t;
}

__global__ void __launch_bounds__(kMseThreads)
    mse_final_kernel(const double* __restrict__ partial, int C, const MseParams p, float* __restrict__ e,
                     float* __restrict__ L) {
  pdl_wait();
  pdl_launch_dependents();
  __shared__ double red[kMseThreads / 32];
  double tot = 0.0;
  const int B = p.B;
  for (int n0 = 0; n0 < B; n0 += kMseThreads) {
    const int n = n0 + threadIdx.x;
    double en = 0.0;
    if (n < B) {
      double s = 0.0;
      for (int c = 0; c < C; ++c) s += partial[static_cast<size_t>(n) * C + c];
      en = s / (static_cast<double>(p.off[n + 1] - p.off[n]) * static_cast<double>(p.d));
      e[n] = static_cast<float>(en);
    }
    tot += block_sum_f64(en, red);
    __syncthreads();
  }
  if (threadIdx.x == 0) *L = static_cast<float>(tot / static_cast<double>(B));
}

}  // namespace

// About four CTAs per SM of a GB300 in all, whatever the device (the
// reduction order, and so the rounding, depends only on B).
int block_mse_chunks(int B) {
  const int want = (608 + B - 1) / B;
  return want < 1 ? 1 : want > 64 ? 64 : want;
}

size_t block_mse_workspace_bytes(int B) {
  return B <= 0 ? 0 : static_cast<size_t>(B) * block_mse_chunks(B) * sizeof(double);
}

cudaError_t launch_block_mse(const uint16_t* Yq, long long ldq, const uint16_t* Yf, long long ldf, const int32_t* off,
                             int B, int d, double* partial, float* e, float* L, cudaStream_t stream) {
  MseParams p;
  p.ldq = ldq;
  p.ldf = ldf;
  p.B = B;
  p.d = d;
  for (int n = 0; n <= B; ++n) p.off[n] = off[n];
  const int C = block_mse_chunks(B);
  cudaError_t err = launch_pdl(mse_partial_kernel, dim3(C, B), dim3(kMseThreads), 0, stream,
                               reinterpret_cast<const __half*>(Yq), reinterpret_cast<const __half*>(Yf), p, partial);
  if (err != cudaSuccess) return err;
  return launch_pdl(mse_final_kernel, dim3(1), dim3(kMseThreads), 0, stream, static_cast<const double*>(partial), C,
                    p, e, L);
}

}  // namespace p4q
