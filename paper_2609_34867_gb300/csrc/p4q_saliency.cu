// CLS-to-patch saliency A_cls (Sec. 3.2 of the paper, Visual Saliency): in
// the vision tower's final self-attention layer each crop's [CLS] token is
// the query; its attention row is the softmax, over the CLS key and the
// crop's patch keys, of q . k / sqrt(d_h), and the saliency of a patch is its
// weight averaged over the heads.
//
// Kernel: one CTA per (image, crop), up to 16 warps each taking heads in
// turn (one warp per head at a time). A token's key row for the head (dh fp16
// values, rows of consecutive tokens H x dh apart) is read by dh / 8 lanes
// with one 16-byte load each, so that a warp load covers whole rows; the
// lanes' partial dot products (fp16 products accumulated in fp32) are summed
// by shuffles. The warp's max and sum then give the head's softmax; the
// per-head weights go to shared memory and are summed over the heads in head
// order (deterministic).
#include <cuda_fp16.h>

#include "p4q.h"
#include "p4q_device.cuh"
#include "p4q_internal.h"

namespace p4q {
namespace {

// Warps per CTA at most (each takes heads warp, warp + warps, ...): 16, so
// that a thread has 128 registers for its head's query and key loads.
constexpr int kMaxWarps = 16;
constexpr int kMaxHeads = 32;

// Lanes that share one token's key row: the row's dh / 8 16-byte chunks, one
// per lane, rounded up to a power of two (idle lanes past the row).
template <int DH>
constexpr int lanes_per_token() {
  return DH / 8 <= 4 ? 4 : DH / 8 <= 8 ? 8 : DH / 8 <= 16 ? 16 : 32;
}

template <int DH>
__global__ void __launch_bounds__(32 * kMaxWarps)
    cls_saliency_kernel(const __half* __restrict__ q_cls, const __half* __restrict__ k_cls,
                        const __half* __restrict__ k, int N, int C, int H, float* __restrict__ A) {
  pdl_wait();
  pdl_launch_dependents();
  constexpr int R = DH / 8;                  // 16-byte chunks per key row
  constexpr int LPT = lanes_per_token<DH>();  // lanes per token
  constexpr int CPL = (R + LPT - 1) / LPT;    // chunks per lane
  constexpr int TPI = 32 / LPT;               // tokens per warp iteration
  extern __shared__ float p[];  // [H][n] softmax weights of the crop's patches per head
  const int b = blockIdx.y, c = blockIdx.x, n = N / C;
  const int lane = threadIdx.x & 31, nwarps = blockDim.x >> 5;
  const int sub = lane % LPT, tok = lane / LPT;
  const float scale = 1.0f / sqrtf(static_cast<float>(DH));
  for (int h = threadIdx.x >> 5; h < H; h += nwarps) {
    const size_t head = (static_cast<size_t>(b) * C + c) * H + h;
    // this lane's chunks of the query, as fp32
    float qf[CPL][8];
    const uint4* q4 = reinterpret_cast<const uint4*>(q_cls + head * DH);
#pragma unroll
    for (int u = 0; u < CPL; ++u) {
      const int ch = sub + u * LPT;
      const uint4 v = ch < R ? q4[ch] : make_uint4(0u, 0u, 0u, 0u);
      const uint32_t w[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        const float2 f = __half22float2(*reinterpret_cast<const __half2*>(&w[e]));
        qf[u][2 * e] = f.x;
        qf[u][2 * e + 1] = f.y;
      }
    }
    // this lane's chunks of a key row (zeros past the row or for no token)
    auto load = [&](const uint4* row, bool live, uint4 (&v)[CPL]) {
#pragma unroll
      for (int u = 0; u < CPL; ++u) {
        const int ch = sub + u * LPT;
        v[u] = (live && ch < R) ? __ldg(row + ch) : make_uint4(0u, 0u, 0u, 0u);
      }
    };
    // partial dot of the loaded chunks, then the sum over the token's lanes
    auto dot = [&](const uint4 (&v)[CPL]) {
      float acc = 0.0f;
#pragma unroll
      for (int u = 0; u < CPL; ++u) {
        const uint32_t w[4] = {v[u].x, v[u].y, v[u].z, v[u].w};
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          const float2 f = __half22float2(*reinterpret_cast<const __half2*>(&w[e]));
          acc = fmaf(qf[u][2 * e], f.x, acc);
          acc = fmaf(qf[u][2 * e + 1], f.y, acc);
        }
      }
#pragma unroll
      for (int o = LPT / 2; o > 0; o >>= 1) acc += __shfl_xor_sync(0xFFFFFFFFu, acc, o);
      return acc;
    };
    uint4 v0[CPL];
    load(reinterpret_cast<const uint4*>(k_cls + head * DH), true, v0);
    const float l0 = dot(v0) * scale;
    float mx = l0;
    float* ph = p + static_cast<size_t>(h) * n;
    constexpr int U = 8;  // token rows in flight per lane
    for (int i0 = 0; i0 < n; i0 += TPI * U) {
      uint4 v[U][CPL];
#pragma unroll
      for (int u = 0; u < U; ++u) {
        const int i = i0 + u * TPI + tok;
        const size_t row = (static_cast<size_t>(b) * N + static_cast<size_t>(c) * n + (i < n ? i : 0)) * H + h;
        load(reinterpret_cast<const uint4*>(k + row * DH), i < n, v[u]);
      }
#pragma unroll
      for (int u = 0; u < U; ++u) {
        const int i = i0 + u * TPI + tok;
        const float l = dot(v[u]) * scale;
        if (i < n) {
          if (sub == 0) ph[i] = l;
          mx = fmaxf(mx, l);
        }
      }
    }
    mx = fmaxf(mx, __shfl_xor_sync(0xFFFFFFFFu, mx, 16));
    mx = fmaxf(mx, __shfl_xor_sync(0xFFFFFFFFu, mx, 8));
    mx = fmaxf(mx, __shfl_xor_sync(0xFFFFFFFFu, mx, 4));
    mx = fmaxf(mx, __shfl_xor_sync(0xFFFFFFFFu, mx, 2));
    mx = fmaxf(mx, __shfl_xor_sync(0xFFFFFFFFu, mx, 1));
    __syncwarp();
    float z = lane == 0 ? expf(l0 - mx) : 0.0f;
    for (int i = lane; i < n; i += 32) {
      const float e = expf(ph[i] - mx);
      ph[i] = e;
      z += e;
    }
    z += __shfl_xor_sync(0xFFFFFFFFu, z, 16);
    z += __shfl_xor_sync(0xFFFFFFFFu, z, 8);
    z += __shfl_xor_sync(0xFFFFFFFFu, z, 4);
    z += __shfl_xor_sync(0xFFFFFFFFu, z, 2);
    z += __shfl_xor_sync(0xFFFFFFFFu, z, 1);
    const float inv = 1.0f / z;
    for (int i = lane; i < n; i += 32) ph[i] *= inv;
  }
  __syncthreads();
  const float invh = 1.0f / static_cast<float>(H);
  for (int i = threadIdx.x; i < n; i += blockDim.x) {
    float s = 0.0f;
    for (int hh = 0; hh < H; ++hh) s += p[static_cast<size_t>(hh) * n + i];
    A[static_cast<size_t>(b) * N + static_cast<size_t>(c) * n + i] = s * invh;
  }
}

template <int DH>
cudaError_t launch_dh(const __half* q_cls, const __half* k_cls, const __half* k, int B, int N, int C, int H,
                      float* A, cudaStream_t stream) {
  const size_t smem = static_cast<size_t>(H) * (N / C) * sizeof(float);
  static size_t smem_set = 48u << 10;
  if (smem > smem_set) {
    cudaError_t e = cudaFuncSetAttribute(cls_saliency_kernel<DH>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         static_cast<int>(smem));
    if (e != cudaSuccess) return e;
    smem_set = smem;
  }
  return launch_pdl(cls_saliency_kernel<DH>, dim3(C, B), dim3(32 * (H < kMaxWarps ? H : kMaxWarps)), smem, stream,
                    q_cls, k_cls, k, N, C, H, A);
}

}  // namespace

size_t cls_saliency_smem_bytes(int N, int C, int H) { return static_cast<size_t>(H) * (N / C) * sizeof(float); }

int cls_saliency_max_heads(int) { return kMaxHeads; }

cudaError_t launch_cls_saliency(const uint16_t* q_cls16, const uint16_t* k_cls16, const uint16_t* k16, int B, int N,
                                int C, int H, int dh, float* A, cudaStream_t stream) {
  const __half* q_cls = reinterpret_cast<const __half*>(q_cls16);
  const __half* k_cls = reinterpret_cast<const __half*>(k_cls16);
  const __half* k = reinterpret_cast<const __half*>(k16);
  switch (dh) {
    case 32: return launch_dh<32>(q_cls, k_cls, k, B, N, C, H, A, stream);
    case 64: return launch_dh<64>(q_cls, k_cls, k, B, N, C, H, A, stream);
    case 80: return launch_dh<80>(q_cls, k_cls, k, B, N, C, H, A, stream);
    case 128: return launch_dh<128>(q_cls, k_cls, k, B, N, C, H, A, stream);
    default: return cudaErrorInvalidValue;
  }
}

}  // namespace p4q
