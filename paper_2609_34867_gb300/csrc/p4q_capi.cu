// The extern "C" boundary of libp4q.so (declared in include/p4q.h): argument
// validation on the host, then the kernel launches of each entry point on the
// caller's stream. Nothing here allocates memory.
#include <cuda_runtime.h>

#include <atomic>
#include <cstdint>
#include <mutex>

#include "p4q.h"
#include "p4q_internal.h"

using namespace p4q;

namespace {

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

std::atomic<uint64_t> g_launches{0};

// Counts one kernel launch when `e` reports success.
cudaError_t counted(cudaError_t e, unsigned int kernels = 1) {
  if (e == cudaSuccess) g_launches.fetch_add(kernels, std::memory_order_relaxed);
  return e;
}

// The kernels are built for sm_103a only; refuse to launch on anything else.
p4q_status check_device() {
  int dev = -1;
  if (cudaGetDevice(&dev) != cudaSuccess) return P4Q_ERR_NO_DEVICE;
  int major = 0, minor = 0;
  if (cudaDeviceGetAttribute(&major, cudaDevAttrComputeCapabilityMajor, dev) != cudaSuccess ||
      cudaDeviceGetAttribute(&minor, cudaDevAttrComputeCapabilityMinor, dev) != cudaSuccess)
    return P4Q_ERR_NO_DEVICE;
  return (major == 10 && minor == 3) ? P4Q_OK : P4Q_ERR_NO_DEVICE;
}

p4q_status from_cuda(cudaError_t e) { return e == cudaSuccess ? P4Q_OK : P4Q_ERR_CUDA; }

struct Budget {
  int Kq, Ks, Kd;
};

// Budget split of Sec. 3.2 in integers; absent signals hand their share to diversity.
Budget split(const p4q_select_params& p, bool have_q, bool have_a) {
  Budget b;
  b.Kq = have_q ? static_cast<int>((static_cast<long long>(p.alpha_permille) * p.K) / 1000) : 0;
  b.Ks = have_a ? static_cast<int>((static_cast<long long>(p.beta_permille) * p.K) / 1000) : 0;
  b.Kd = p.K - b.Kq - b.Ks;
  return b;
}

p4q_status check_select_args(const uint16_t* V, int B, int N, int d, int J, const p4q_select_params* params,
                             const int32_t* idx) {
  if (!V || !params || !idx || B < 1 || N < 1 || d < 1 || J < 0) return P4Q_ERR_INVALID_ARG;
  if (params->K < 1 || params->K > N || params->alpha_permille < 0 || params->beta_permille < 0 ||
      params->alpha_permille + params->beta_permille > 1000)
    return P4Q_ERR_INVALID_ARG;
  if (N > P4Q_MAX_TOKENS || J > P4Q_MAX_CONCEPTS || d % 128 != 0 || d > P4Q_MAX_ROW || B > 65535)
    return P4Q_ERR_UNSUPPORTED_SHAPE;
  if (!aligned16(V) || !aligned16(idx)) return P4Q_ERR_MISALIGNED;
  return P4Q_OK;
}

// A second stream of the library per device, with a fork and a join event,
// on which the selector's token-pair GEMM (Gram mode) runs beside the
// concept, query and stage-1/2 launches; created on the first call that is
// not being captured into a graph. Its users hold g_side_mutex from the fork
// to the join (the events are shared).
struct SideStream {
  cudaStream_t s = nullptr;
  cudaEvent_t fork = nullptr, join = nullptr;
  bool failed = false;
};
std::mutex g_side_mutex;
SideStream g_side[64];

SideStream* side_stream(cudaStream_t stream) {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return nullptr;
  SideStream& r = g_side[dev];
  if (r.s) return &r;
  if (r.failed) return nullptr;
  cudaStreamCaptureStatus cs = cudaStreamCaptureStatusNone;
  if (cudaStreamIsCapturing(stream, &cs) != cudaSuccess || cs != cudaStreamCaptureStatusNone) return nullptr;
  if (cudaStreamCreateWithFlags(&r.s, cudaStreamNonBlocking) != cudaSuccess ||
      cudaEventCreateWithFlags(&r.fork, cudaEventDisableTiming) != cudaSuccess ||
      cudaEventCreateWithFlags(&r.join, cudaEventDisableTiming) != cudaSuccess) {
    cudaGetLastError();
    r.failed = true;  // the serial order is used from now on
    r.s = nullptr;
    return nullptr;
  }
  return &r;
}

// R0 = Kq + Ks of a call (the workspace layout depends on it).
int select_r0(const p4q_select_params& p, bool have_q, bool have_a) {
  const Budget bud = split(p, have_q, have_a);
  return bud.Kq + bud.Ks;
}

// The selector: fake-quantized copies of the concepts and of the tokens with
// the query dot products (in the token pass, or a narrow GEMM), stages 1-2, the initial diversity maxima on
// the tensor cores (Gram mode: one GEMM of all token pairs; otherwise R0's
// expanded codes gathered, a GEMM against every token and a row pass, then
// the candidates' pairwise GEMM), stage 3 (writes idx). Work is ordered on
// `stream`; with use_side the Gram GEMM runs on the library's second stream,
// forked from and joined back into `stream`.
p4q_status run_select(const uint16_t* V, int B, int N, int d, const uint16_t* Q, int J, const float* A_cls,
                      const p4q_select_params* params, int32_t* idx, void* ws, size_t ws_bytes,
                      cudaStream_t stream, bool use_side = true) {
  const bool have_q = (Q != nullptr && J > 0);
  const int Jeff = have_q ? J : 0;
  if (have_q && !aligned16(Q)) return P4Q_ERR_MISALIGNED;
  if (A_cls && !aligned16(A_cls)) return P4Q_ERR_MISALIGNED;
  const Budget bud = split(*params, have_q, A_cls != nullptr);
  const int R0 = bud.Kq + bud.Ks;
  const bool gram = select_gram_mode(N, bud.Kd);
  const int C = select_candidates(N, R0, bud.Kd);
  const size_t need = select_workspace_layout(B, N, d, Jeff, R0, C, gram, nullptr, nullptr);
  if (!ws || ws_bytes < need) return P4Q_ERR_WORKSPACE_TOO_SMALL;
  if ((reinterpret_cast<uintptr_t>(ws) & 255u) != 0) return P4Q_ERR_MISALIGNED;
  SelectWorkspace w;
  select_workspace_layout(B, N, d, Jeff, R0, C, gram, &w, ws);
  SelectPlan plan{B, N, d, Jeff, params->K, bud.Kq, bud.Ks, bud.Kd};

  // Fake-quantized copies of the concepts, then of the projector features:
  // the codes expanded to one byte each (what the tensor-core stages read),
  // their row sums and squared norms, and the code dot products of every
  // token with its image's concepts (the query cosines are taken from them
  // in stages 1-2): in the token pass itself where it applies, else on the
  // tensor cores after it.
  cudaError_t e;
  const int Jq = bud.Kq > 0 ? Jeff : 0;  // concepts whose dot products stage 1 reads
  if (Jq > 0) {
    RowSource qsrc;
    qsrc.X = Q;
    RowSinks oq;
    oq.codes = w.qcodes;
    oq.scale = w.qscale;
    oq.norm2 = w.qnorm;
    oq.u = w.qu;
    oq.sum_u = w.qsum;
    if ((e = counted(launch_quant_rows(qsrc, B * Jeff, d, oq, stream))) != cudaSuccess) return from_cuda(e);
  }
  RowSinks sv;
  sv.scale = w.vscale;
  sv.norm2 = w.vnorm;
  sv.u = w.vu;
  sv.sum_u = w.vsum;
  if (select_token_quant_applies(d, Jq)) {
    if ((e = counted(launch_select_token_quant(V, B, N, d, Jq, w.qu, w.qsum, sv, w.qdots, w.q_pitch, stream))) !=
        cudaSuccess)
      return from_cuda(e);
  } else {
    RowSource src;
    src.X = V;
    if ((e = counted(launch_quant_rows(src, B * N, d, sv, stream))) != cudaSuccess) return from_cuda(e);
    if (Jq > 0 && (e = counted(launch_query_dots(plan, w, stream))) != cudaSuccess) return from_cuda(e);
  }
  // Gram mode: the token-pair GEMM needs only the token codes; it runs on the
  // library's second stream beside the stage-1/2 launch
  std::unique_lock<std::mutex> side_lock(g_side_mutex, std::defer_lock);
  SideStream* side = nullptr;
  if (w.gram && use_side) {
    side_lock.lock();
    side = side_stream(stream);
    if (side) {
      cudaError_t se = cudaEventRecord(side->fork, stream);
      if (se == cudaSuccess) se = cudaStreamWaitEvent(side->s, side->fork, 0);
      if (se == cudaSuccess) se = counted(launch_gram(plan, w, side->s));
      if (se == cudaSuccess) se = cudaEventRecord(side->join, side->s);
      if (se != cudaSuccess) return from_cuda(se);
    } else {
      side_lock.unlock();
    }
  }
  if (R0 > 0 || bud.Kd > 0) {
    // stages 1-2 (also the bits of an empty R0, and idx when Kd = 0)
    if ((e = counted(launch_select_stages12(plan, w, A_cls, idx, stream))) != cudaSuccess) return from_cuda(e);
  }
  if (bud.Kd == 0) return P4Q_OK;
  if (w.gram) {
    // small images: every token pair's dot product; stage 3 takes R0's maxima from it
    if (side) {
      if ((e = cudaStreamWaitEvent(stream, side->join, 0)) != cudaSuccess) return from_cuda(e);
    } else if ((e = counted(launch_gram(plan, w, stream))) != cudaSuccess) {
      return from_cuda(e);
    }
    if (R0 > 0 && (e = counted(launch_gram_cosmax(plan, w, stream))) != cudaSuccess) return from_cuda(e);
  } else {
    if (R0 > 0) {
      if ((e = counted(launch_gather_r0(plan, w, stream))) != cudaSuccess) return from_cuda(e);
      // one GEMM with the cosine-max epilogue, or (R0 > kCosMaxCols) a GEMM and a row pass
      if ((e = counted(launch_r0_cosmax(plan, w, stream), R0 <= kCosMaxCols ? 1 : 2)) != cudaSuccess)
        return from_cuda(e);
    }
    // candidates, their rows, their pairwise dot products
    if ((e = counted(launch_candidates(plan, w, stream), 3)) != cudaSuccess) return from_cuda(e);
  }
  return from_cuda(counted(launch_select_diverse(plan, w, idx, stream)));
}

p4q_status check_rows(const void* X, int M, int Kin, const void* Xq, const void* s) {
  if (M < 0 || Kin < 1) return P4Q_ERR_INVALID_ARG;
  if (M > 0 && (!X || !Xq || !s)) return P4Q_ERR_INVALID_ARG;
  if (Kin % 16 != 0 || Kin > P4Q_MAX_ROW) return P4Q_ERR_UNSUPPORTED_SHAPE;
  if (M > 0 && (!aligned16(X) || !aligned16(Xq) || !aligned16(s))) return P4Q_ERR_MISALIGNED;
  return P4Q_OK;
}

p4q_status check_gemm(const void* Xq, int M, int Kin, const void* Wq, int N, const void* out) {
  if (M < 0 || N < 1 || Kin < 1 || !Wq || (M > 0 && (!Xq || !out))) return P4Q_ERR_INVALID_ARG;
  if (Kin % 128 != 0 || Kin > P4Q_MAX_ROW || N % 8 != 0 || M > 65535 * 128) return P4Q_ERR_UNSUPPORTED_SHAPE;
  if (!aligned16(Wq) || (M > 0 && (!aligned16(Xq) || !aligned16(out)))) return P4Q_ERR_MISALIGNED;
  return P4Q_OK;
}

}  // namespace

extern "C" {

const char* p4q_status_string(p4q_status s) {
  switch (s) {
    case P4Q_OK: return "ok";
    case P4Q_ERR_INVALID_ARG: return "invalid argument";
    case P4Q_ERR_UNSUPPORTED_SHAPE: return "unsupported shape";
    case P4Q_ERR_MISALIGNED: return "device pointer not 16-byte aligned";
    case P4Q_ERR_WORKSPACE_TOO_SMALL: return "workspace too small";
    case P4Q_ERR_CUDA: return "CUDA error";
    case P4Q_ERR_TIMEOUT: return "a bounded device wait timed out";
    case P4Q_ERR_NO_DEVICE: return "no sm_103 device is current";
  }
  return "unknown status";
}

uint64_t p4q_launch_count(void) { return g_launches.load(std::memory_order_relaxed); }

p4q_status p4q_cls_saliency(const uint16_t* q_cls, const uint16_t* k_cls, const uint16_t* k, int B, int N, int C,
                            int H, int dh, float* A_cls, p4q_stream_t stream) {
  if (!q_cls || !k_cls || !k || !A_cls || B < 1 || N < 1 || C < 1 || H < 1) return P4Q_ERR_INVALID_ARG;
  if (B > 65535 || N % C != 0 || N / C > P4Q_MAX_TOKENS || (dh != 32 && dh != 64 && dh != 80 && dh != 128) ||
      H > cls_saliency_max_heads(dh) || cls_saliency_smem_bytes(N, C, H) > 227u * 1024u)
    return P4Q_ERR_UNSUPPORTED_SHAPE;
  if (!aligned16(q_cls) || !aligned16(k_cls) || !aligned16(k) || !aligned16(A_cls)) return P4Q_ERR_MISALIGNED;
  p4q_status st = check_device();
  if (st != P4Q_OK) return st;
  return from_cuda(counted(launch_cls_saliency(q_cls, k_cls, k, B, N, C, H, dh, A_cls,
                                               reinterpret_cast<cudaStream_t>(stream))));
}

p4q_status p4q_set_gemm_variant(int variant) {
  if (variant < 0 || variant > 3) return P4Q_ERR_INVALID_ARG;
  set_gemm_pair_mode(variant == 0 || variant == 3 ? -1 : variant == 1 ? 0 : 1);
  set_gemm8_mode(variant == 0 ? 0 : variant == 3 ? 2 : 1);
  return P4Q_OK;
}

p4q_status p4q_device_status(p4q_stream_t stream) {
  if (cudaStreamSynchronize(reinterpret_cast<cudaStream_t>(stream)) != cudaSuccess) return P4Q_ERR_CUDA;
  const unsigned int g = gemm_read_and_clear_error() | gemm8_read_and_clear_error() | quant_read_and_clear_error() |
                         attn_read_and_clear_error() | peak_read_and_clear_error() | diverse_read_and_clear_error();
  if (cudaGetLastError() != cudaSuccess) return P4Q_ERR_CUDA;
  return g ? P4Q_ERR_TIMEOUT : P4Q_OK;
}

p4q_status p4q_test_wait_timeout(uint32_t limit_us, p4q_stream_t stream) {
  if (limit_us < 1u || limit_us > 1000000u) return P4Q_ERR_INVALID_ARG;
  p4q_status st = check_device();
  if (st != P4Q_OK) return st;
  return from_cuda(counted(launch_expired_wait(1000ull * limit_us, reinterpret_cast<cudaStream_t>(stream))));
}

p4q_status p4q_peak_probe(int kind, int iters, uint32_t* sink, double* ops, p4q_stream_t stream) {
  if (kind < 0 || kind > 2 || iters < 1 || iters > (1 << 24) || !sink || !ops) return P4Q_ERR_INVALID_ARG;
  if (!aligned16(sink)) return P4Q_ERR_MISALIGNED;
  p4q_status st = check_device();
  if (st != P4Q_OK) return st;
  if (static_cast<size_t>(num_sms()) * 4 > peak_probe_sink_words()) return P4Q_ERR_UNSUPPORTED_SHAPE;
  return from_cuda(counted(launch_peak_probe(kind, iters, sink, ops, reinterpret_cast<cudaStream_t>(stream))));
}

p4q_status p4q_quant_act(const uint16_t* X, int M, int Kin, uint8_t* Xq, float* s_a, p4q_stream_t stream) {
  return p4q_quant_act_ld(X, Kin, M, Kin, Xq, s_a, stream);
}

p4q_status p4q_quant_act_expanded(const uint16_t* X, int ldx, int M, int Kin, uint8_t* Xq, float* s_a, uint8_t* Xu,
                                  int32_t* sum_xu, p4q_stream_t stream) {
  p4q_status st = check_rows(X, M, Kin, Xq, s_a);
  if (st != P4Q_OK) return st;
  if (ldx < Kin || (M > 0 && (!Xu || !sum_xu))) return P4Q_ERR_INVALID_ARG;
  if (ldx % 8 != 0 || (M > 0 && (!aligned16(Xu) || !aligned16(sum_xu)))) return P4Q_ERR_MISALIGNED;
  if (M == 0) return P4Q_OK;
  if ((st = check_device()) != P4Q_OK) return st;
  RowSource src;
  src.X = X;
  src.ldx = ldx;
  RowSinks o;
  o.codes = Xq;
  o.scale = s_a;
  o.u = Xu;
  o.sum_u = sum_xu;
  return from_cuda(counted(launch_quant_rows(src, M, Kin, o, reinterpret_cast<cudaStream_t>(stream))));
}

p4q_status p4q_swiglu_quant_expanded(const uint16_t* gate, int ld_gate, const uint16_t* up, int ld_up, int M, int Kin,
                                     uint8_t* Xq, float* s_a, uint8_t* Xu, int32_t* sum_xu, p4q_stream_t stream) {
  if (M < 0 || Kin < 16 || ld_gate < Kin || ld_up < Kin || (!Xu) != (!sum_xu)) return P4Q_ERR_INVALID_ARG;
  if (M > 0 && (!gate || !up || !Xq || !s_a)) return P4Q_ERR_INVALID_ARG;
  if (Kin % 16 != 0 || Kin > P4Q_MAX_ROW) return P4Q_ERR_UNSUPPORTED_SHAPE;
  if (ld_gate % 8 != 0 || ld_up % 8 != 0) return P4Q_ERR_MISALIGNED;
  if (M > 0 && (!aligned16(gate) || !aligned16(up) || !aligned16(Xq) || !aligned16(s_a) ||
                (Xu && (!aligned16(Xu) || !aligned16(sum_xu)))))
    return P4Q_ERR_MISALIGNED;
  if (M == 0) return P4Q_OK;
  p4q_status st = check_device();
  if (st != P4Q_OK) return st;
  return from_cuda(counted(launch_swiglu_quant(gate, ld_gate, up, ld_up, M, Kin, Xq, s_a, Xu, sum_xu,
                                               reinterpret_cast<cudaStream_t>(stream))));
}

p4q_status p4q_rmsnorm_quant_expanded(const uint16_t* X, int ldx, const uint16_t* w, float eps, int M, int Kin,
                                      uint8_t* Xq, float* s_a, uint8_t* Xu, int32_t* sum_xu, p4q_stream_t stream) {
  if (M < 0 || Kin < 16 || ldx < Kin || (!Xu) != (!sum_xu) || !(eps >= 0.0f) || !(eps < INFINITY))
    return P4Q_ERR_INVALID_ARG;
  if (M > 0 && (!X || !w || !Xq || !s_a)) return P4Q_ERR_INVALID_ARG;
  if (Kin % 16 != 0 || Kin > P4Q_MAX_ROW) return P4Q_ERR_UNSUPPORTED_SHAPE;
  if (ldx % 8 != 0) return P4Q_ERR_MISALIGNED;
  if (M > 0 && (!aligned16(X) || !aligned16(w) || !aligned16(Xq) || !aligned16(s_a) ||
                (Xu && (!aligned16(Xu) || !aligned16(sum_xu)))))
    return P4Q_ERR_MISALIGNED;
  if (M == 0) return P4Q_OK;
  p4q_status st = check_device();
  if (st != P4Q_OK) return st;
  return from_cuda(counted(launch_rmsnorm_quant(X, ldx, w, eps, M, Kin, Xq, s_a, Xu, sum_xu,
                                                reinterpret_cast<cudaStream_t>(stream))));
}

p4q_status p4q_causal_attention(const uint16_t* q, int ldq, const uint16_t* k, int ldk, const uint16_t* v, int ldv,
                                int B, int m, int H, int Hkv, int dh, uint16_t* o, int ldo, p4q_stream_t stream) {
  if (B < 0 || m < 1 || H < 1 || Hkv < 1 || H % Hkv != 0) return P4Q_ERR_INVALID_ARG;
  if (ldq < H * dh || ldk < Hkv * dh || ldv < Hkv * dh || ldo < H * dh) return P4Q_ERR_INVALID_ARG;
  if (B > 0 && (!q || !k || !v || !o)) return P4Q_ERR_INVALID_ARG;
  if (dh != 128 || m > kAttnMaxLen || B > 65535 || H > 65535 || static_cast<long long>(B) * m > (1ll << 31) - 1)
    return P4Q_ERR_UNSUPPORTED_SHAPE;
  if (ldq % 8 != 0 || ldk % 8 != 0 || ldv % 8 != 0 || ldo % 8 != 0) return P4Q_ERR_MISALIGNED;
  if (B > 0 && (!aligned16(q) || !aligned16(k) || !aligned16(v) || !aligned16(o))) return P4Q_ERR_MISALIGNED;
  if (B == 0) return P4Q_OK;
  p4q_status st = check_device();
  if (st != P4Q_OK) return st;
  return from_cuda(counted(launch_causal_attention(q, ldq, k, ldk, v, ldv, B, m, H, Hkv, o, ldo,
                                                   reinterpret_cast<cudaStream_t>(stream))));
}

size_t p4q_block_mse_workspace_bytes(int B) {
  return (B < 1 || B > kMseMaxSamples) ? 0 : block_mse_workspace_bytes(B);
}

p4q_status p4q_block_mse(const uint16_t* Yq, int ldq, const uint16_t* Yf, int ldf, const int32_t* offsets, int B,
                         int d, float* e, float* L, void* ws, size_t ws_bytes, p4q_stream_t stream) {
  if (!Yq || !Yf || !offsets || !e || !L || B < 1 || d < 8 || ldq < d || ldf < d) return P4Q_ERR_INVALID_ARG;
  if (B > kMseMaxSamples) return P4Q_ERR_UNSUPPORTED_SHAPE;
  if (offsets[0] != 0) return P4Q_ERR_INVALID_ARG;
  for (int n = 0; n < B; ++n)
    if (offsets[n + 1] <= offsets[n]) return P4Q_ERR_INVALID_ARG;
  if (d % 8 != 0) return P4Q_ERR_UNSUPPORTED_SHAPE;
  if (ldq % 8 != 0 || ldf % 8 != 0 || !aligned16(Yq) || !aligned16(Yf) || !aligned16(ws)) return P4Q_ERR_MISALIGNED;
  if (!ws || ws_bytes < block_mse_workspace_bytes(B)) return P4Q_ERR_WORKSPACE_TOO_SMALL;
  p4q_status st = check_device();
  if (st != P4Q_OK) return st;
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  return from_cuda(counted(launch_block_mse(Yq, ldq, Yf, ldf, offsets, B, d, static_cast<double*>(ws), e, L, s), 2));
}

p4q_status p4q_topk_replacement(const float* s_ref, const float* s_alt, int B, int N, int K, int32_t* inter,
                                float* rho, p4q_stream_t stream) {
  if (B < 0 || N < 1 || K < 1 || K > N) return P4Q_ERR_INVALID_ARG;
  if (B > 0 && (!s_ref || !s_alt || !inter || !rho)) return P4Q_ERR_INVALID_ARG;
  if (N > P4Q_MAX_TOKENS || B > 65535) return P4Q_ERR_UNSUPPORTED_SHAPE;
  if (B == 0) return P4Q_OK;
  p4q_status st = check_device();
  if (st != P4Q_OK) return st;
  return from_cuda(
      counted(launch_topk_replacement(s_ref, s_alt, B, N, K, inter, rho, reinterpret_cast<cudaStream_t>(stream))));
}

p4q_status p4q_quant_act_ld(const uint16_t* X, int ldx, int M, int Kin, uint8_t* Xq, float* s_a,
                            p4q_stream_t stream) {
  p4q_status st = check_rows(X, M, Kin, Xq, s_a);
  if (st != P4Q_OK) return st;
  if (ldx < Kin) return P4Q_ERR_INVALID_ARG;
  if (ldx % 8 != 0) return P4Q_ERR_MISALIGNED;
  if (M == 0) return P4Q_OK;
  if ((st = check_device()) != P4Q_OK) return st;
  RowSource src;
  src.X = X;
  src.ldx = ldx;
  RowSinks o;
  o.codes = Xq;
  o.scale = s_a;
  return from_cuda(counted(launch_quant_rows(src, M, Kin, o, reinterpret_cast<cudaStream_t>(stream))));
}

p4q_status p4q_quant_weight(const uint16_t* W, int N, int Kin, uint8_t* Wq, float* s_w, p4q_stream_t stream) {
  return p4q_quant_act(W, N, Kin, Wq, s_w, stream);
}

p4q_status p4q_w4a4_linear(const uint8_t* Xq, const float* s_a, int M, int Kin, const uint8_t* Wq,
                           const float* s_w, int N, uint16_t* Y, p4q_stream_t stream) {
  p4q_status st = check_gemm(Xq, M, Kin, Wq, N, Y);
  if (st != P4Q_OK) return st;
  if (!s_w || (M > 0 && !s_a)) return P4Q_ERR_INVALID_ARG;
  if (M == 0) return P4Q_OK;
  if ((st = check_device()) != P4Q_OK) return st;
  GemmArgs g;
  g.A = Xq;
  g.B = Wq;
  g.M = M;
  g.N = N;
  g.K = Kin;
  g.out = GemmOut::kHalf;
  g.D = Y;
  g.s_a = s_a;
  g.s_b = s_w;
  return from_cuda(counted(launch_w4a4_gemm(g, reinterpret_cast<cudaStream_t>(stream))));
}

size_t p4q_w4a4_linear_workspace_bytes(int M, int N, int Kin) {
  if (M < 0 || N < 1 || Kin < 1 || Kin % 128 != 0 || Kin > P4Q_MAX_ROW || N % 8 != 0) return 0;
  return gemm8_workspace_bytes(M, N, Kin);
}

namespace {

// The workspace entry points: the expanded-operand path when a workspace is
// given and the shape qualifies, else the in-kernel unpack.
p4q_status run_linear_ws(const GemmArgs& g, void* ws, size_t ws_bytes, cudaStream_t stream) {
  if (ws) {
    if (!aligned16(ws)) return P4Q_ERR_MISALIGNED;
    if (ws_bytes < gemm8_workspace_bytes(g.M, g.N, g.K)) return P4Q_ERR_WORKSPACE_TOO_SMALL;
    if (gemm8_applies(g)) return from_cuda(counted(launch_w4a4_gemm8(g, ws, ws_bytes, stream), 3));
  }
  return from_cuda(counted(launch_w4a4_gemm(g, stream)));
}

}  // namespace

p4q_status p4q_w4a4_linear_ws(const uint8_t* Xq, const float* s_a, int M, int Kin, const uint8_t* Wq,
                              const float* s_w, int N, uint16_t* Y, void* ws, size_t ws_bytes, p4q_stream_t stream) {
  p4q_status st = check_gemm(Xq, M, Kin, Wq, N, Y);
  if (st != P4Q_OK) return st;
  if (!s_w || (M > 0 && !s_a)) return P4Q_ERR_INVALID_ARG;
  if (M == 0) return P4Q_OK;
  if ((st = check_device()) != P4Q_OK) return st;
  GemmArgs g;
  g.A = Xq;
  g.B = Wq;
  g.M = M;
  g.N = N;
  g.K = Kin;
  g.out = GemmOut::kHalf;
  g.D = Y;
  g.s_a = s_a;
  g.s_b = s_w;
  return run_linear_ws(g, ws, ws_bytes, reinterpret_cast<cudaStream_t>(stream));
}

p4q_status p4q_w4a4_gemm_s32_ws(const uint8_t* Xq, int M, int Kin, const uint8_t* Wq, int N, int32_t* acc, void* ws,
                                size_t ws_bytes, p4q_stream_t stream) {
  p4q_status st = check_gemm(Xq, M, Kin, Wq, N, acc);
  if (st != P4Q_OK || M == 0) return st;
  if ((st = check_device()) != P4Q_OK) return st;
  GemmArgs g;
  g.A = Xq;
  g.B = Wq;
  g.M = M;
  g.N = N;
  g.K = Kin;
  g.out = GemmOut::kS32;
  g.D = acc;
  return run_linear_ws(g, ws, ws_bytes, reinterpret_cast<cudaStream_t>(stream));
}

p4q_status p4q_expand_codes(const uint8_t* q, int rows, int Kin, uint8_t* u, int32_t* sum_u, p4q_stream_t stream) {
  if (rows < 0 || Kin < 1) return P4Q_ERR_INVALID_ARG;
  if (rows > 0 && (!q || !u || !sum_u)) return P4Q_ERR_INVALID_ARG;
  if (Kin % 128 != 0 || Kin > P4Q_MAX_ROW) return P4Q_ERR_UNSUPPORTED_SHAPE;
  if (rows > 0 && (!aligned16(q) || !aligned16(u) || !aligned16(sum_u))) return P4Q_ERR_MISALIGNED;
  if (rows == 0) return P4Q_OK;
  p4q_status st = check_device();
  if (st != P4Q_OK) return st;
  return from_cuda(counted(launch_expand_codes(q, rows, Kin, u, sum_u, reinterpret_cast<cudaStream_t>(stream))));
}

p4q_status p4q_w4a4_linear_expanded(const uint8_t* Xu, const int32_t* sum_xu, const float* s_a, int M, int Kin,
                                    const uint8_t* Wu, const int32_t* sum_wu, const float* s_w, int N, uint16_t* Y,
                                    p4q_stream_t stream) {
  if (M < 0 || N < 1 || Kin < 1 || !Wu || !sum_wu || !s_w || (M > 0 && (!Xu || !sum_xu || !s_a || !Y)))
    return P4Q_ERR_INVALID_ARG;
  if (Kin % 128 != 0 || Kin > P4Q_MAX_ROW || N % 8 != 0 || N < 256) return P4Q_ERR_UNSUPPORTED_SHAPE;
  if (!aligned16(Wu) || (M > 0 && (!aligned16(Xu) || !aligned16(Y)))) return P4Q_ERR_MISALIGNED;
  if (M == 0) return P4Q_OK;
  p4q_status st = check_device();
  if (st != P4Q_OK) return st;
  GemmArgs g;
  g.M = M;
  g.N = N;
  g.K = Kin;
  g.out = GemmOut::kHalf;
  g.D = Y;
  g.s_a = s_a;
  g.s_b = s_w;
  return from_cuda(counted(launch_gemm8(g, Xu, sum_xu, Wu, sum_wu, reinterpret_cast<cudaStream_t>(stream))));
}

p4q_status p4q_w4a4_linear_expanded_rowmax(const uint8_t* Xu, const int32_t* sum_xu, const float* s_a, int M,
                                           int Kin, const uint8_t* Wu, const int32_t* sum_wu, const float* s_w, int N,
                                           uint16_t* Y, int nblk, const int* col0, const int* ncols,
                                           uint32_t* rowmax, p4q_stream_t stream) {
  if (M < 0 || N < 1 || Kin < 1 || !Wu || !sum_wu || !s_w || (M > 0 && (!Xu || !sum_xu || !s_a || !Y)))
    return P4Q_ERR_INVALID_ARG;
  if (nblk < 1 || nblk > 2 || !col0 || !ncols || (M > 0 && !rowmax)) return P4Q_ERR_INVALID_ARG;
  for (int b = 0; b < nblk; ++b) {
    if (col0[b] < 0 || ncols[b] < 1 || col0[b] > N - ncols[b]) return P4Q_ERR_INVALID_ARG;
    if (col0[b] % 32 != 0 || ncols[b] % 32 != 0) return P4Q_ERR_UNSUPPORTED_SHAPE;
  }
  if (Kin % 128 != 0 || Kin > P4Q_MAX_ROW || N % 8 != 0 || N < 256) return P4Q_ERR_UNSUPPORTED_SHAPE;
  if (!aligned16(Wu) || (M > 0 && (!aligned16(Xu) || !aligned16(Y) || !aligned16(rowmax)))) return P4Q_ERR_MISALIGNED;
  if (M == 0) return P4Q_OK;
  p4q_status st = check_device();
  if (st != P4Q_OK) return st;
  cudaStream_t cs = reinterpret_cast<cudaStream_t>(stream);
  cudaError_t e = cudaMemsetAsync(rowmax, 0, sizeof(uint32_t) * static_cast<size_t>(nblk) * M, cs);
  if (e != cudaSuccess) return from_cuda(e);
  GemmArgs g;
  g.M = M;
  g.N = N;
  g.K = Kin;
  g.out = GemmOut::kHalf;
  g.D = Y;
  g.s_a = s_a;
  g.s_b = s_w;
  g.rowmax = rowmax;
  g.rm_n = nblk;
  for (int b = 0; b < nblk; ++b) {
    g.rm_c0[b] = col0[b];
    g.rm_c1[b] = col0[b] + ncols[b];
  }
  return from_cuda(counted(launch_gemm8(g, Xu, sum_xu, Wu, sum_wu, cs)));
}

p4q_status p4q_quant_act_expanded_rowmax(const uint16_t* Y, int ldy, int M, int nblk, const int* col0,
                                         const int* ncols, const uint32_t* rowmax, uint8_t* const* Xq,
                                         float* const* s_a, uint8_t* const* Xu, int32_t* const* sum_xu,
                                         p4q_stream_t stream) {
  if (M < 0 || nblk < 1 || nblk > 2 || !col0 || !ncols || !s_a || !Xu || !sum_xu) return P4Q_ERR_INVALID_ARG;
  if (M > 0 && (!Y || !rowmax)) return P4Q_ERR_INVALID_ARG;
  RowmaxBlock blk[2];
  for (int b = 0; b < nblk; ++b) {
    if (col0[b] < 0 || ncols[b] < 1 || ldy < ncols[b] || col0[b] > ldy - ncols[b]) return P4Q_ERR_INVALID_ARG;
    if (ncols[b] % 256 != 0 || ncols[b] > P4Q_MAX_ROW) return P4Q_ERR_UNSUPPORTED_SHAPE;
    if (col0[b] % 8 != 0) return P4Q_ERR_MISALIGNED;
    if (M > 0 && (!s_a[b] || !Xu[b] || !sum_xu[b])) return P4Q_ERR_INVALID_ARG;
    if (M > 0 && (!aligned16(s_a[b]) || !aligned16(Xu[b]) || !aligned16(sum_xu[b]) ||
                  (Xq && Xq[b] && !aligned16(Xq[b]))))
      return P4Q_ERR_MISALIGNED;
    blk[b].col0 = col0[b];
    blk[b].L = ncols[b];
    blk[b].codes = Xq ? Xq[b] : nullptr;
    blk[b].scale = M > 0 ? s_a[b] : nullptr;
    blk[b].u = M > 0 ? Xu[b] : nullptr;
    blk[b].sum_u = M > 0 ? sum_xu[b] : nullptr;
  }
  if (ldy % 8 != 0 || (M > 0 && (!aligned16(Y) || !aligned16(rowmax)))) return P4Q_ERR_MISALIGNED;
  if (M == 0) return P4Q_OK;
  p4q_status st = check_device();
  if (st != P4Q_OK) return st;
  return from_cuda(counted(launch_quant_rowmax(Y, ldy, M, nblk, blk, rowmax, reinterpret_cast<cudaStream_t>(stream))));
}

p4q_status p4q_w4a4_gemm_s32(const uint8_t* Xq, int M, int Kin, const uint8_t* Wq, int N, int32_t* acc,
                             p4q_stream_t stream) {
  p4q_status st = check_gemm(Xq, M, Kin, Wq, N, acc);
  if (st != P4Q_OK || M == 0) return st;
  if ((st = check_device()) != P4Q_OK) return st;
  GemmArgs g;
  g.A = Xq;
  g.B = Wq;
  g.M = M;
  g.N = N;
  g.K = Kin;
  g.out = GemmOut::kS32;
  g.D = acc;
  return from_cuda(counted(launch_w4a4_gemm(g, reinterpret_cast<cudaStream_t>(stream))));
}

size_t p4q_select_workspace_bytes(int B, int N, int d, int J, const p4q_select_params* params) {
  if (!params || B < 1 || N < 1 || d < 1 || J < 0 || N > P4Q_MAX_TOKENS || J > P4Q_MAX_CONCEPTS ||
      d % 128 != 0 || d > P4Q_MAX_ROW || params->K < 1 || params->K > N)
    return 0;
  // every region at the largest a call with these sizes can need: R0 with
  // concepts and CLS saliency present, the candidates with both absent (K_d = K)
  const bool gram = select_gram_mode(N, params->K);
  return select_workspace_layout(B, N, d, J, select_r0(*params, J > 0, true), select_candidates(N, 0, params->K),
                                 gram, nullptr, nullptr);
}

p4q_status p4q_select(const uint16_t* V, int B, int N, int d, const uint16_t* Q, int J, const float* A_cls,
                      const p4q_select_params* params, int32_t* idx, void* ws, size_t ws_bytes,
                      p4q_stream_t stream) {
  p4q_status st = check_select_args(V, B, N, d, J, params, idx);
  if (st != P4Q_OK) return st;
  if ((st = check_device()) != P4Q_OK) return st;
  return run_select(V, B, N, d, Q, J, A_cls, params, idx, ws, ws_bytes, reinterpret_cast<cudaStream_t>(stream));
}

p4q_status p4q_select_gather_quant(const uint16_t* V, int B, int N, int d, const uint16_t* Q, int J,
                                   const float* A_cls, const uint16_t* text, int T,
                                   const p4q_select_params* params, int32_t* idx, uint16_t* X, uint8_t* Xq,
                                   float* s_a, void* ws, size_t ws_bytes, p4q_stream_t stream) {
  return p4q_select_gather_quant_expanded(V, B, N, d, Q, J, A_cls, text, T, params, idx, X, Xq, s_a, nullptr,
                                          nullptr, ws, ws_bytes, stream);
}

p4q_status p4q_select_gather_quant_expanded(const uint16_t* V, int B, int N, int d, const uint16_t* Q, int J,
                                            const float* A_cls, const uint16_t* text, int T,
                                            const p4q_select_params* params, int32_t* idx, uint16_t* X,
                                            uint8_t* Xq, float* s_a, uint8_t* Xu, int32_t* sum_xu, void* ws,
                                            size_t ws_bytes, p4q_stream_t stream) {
  p4q_status st = check_select_args(V, B, N, d, J, params, idx);
  if (st != P4Q_OK) return st;
  // the packed codes may be left out when the expanded ones are written
  if (T < 0 || (T > 0 && !text) || !X || (!Xq && !Xu) || !s_a || (!Xu != !sum_xu)) return P4Q_ERR_INVALID_ARG;
  if ((T > 0 && !aligned16(text)) || !aligned16(X) || (Xq && !aligned16(Xq)) || !aligned16(s_a))
    return P4Q_ERR_MISALIGNED;
  if (Xu && (!aligned16(Xu) || !aligned16(sum_xu))) return P4Q_ERR_MISALIGNED;
  if ((st = check_device()) != P4Q_OK) return st;
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  st = run_select(V, B, N, d, Q, J, A_cls, params, idx, ws, ws_bytes, s);
  if (st != P4Q_OK) return st;
  // Gather the FP16 originals of the kept tokens, then the text rows, and
  // quantize every row of the pruned sequence.
  RowSource src;
  src.X = V;
  src.idx = idx;
  src.text = text;
  src.N = N;
  src.K = params->K;
  src.T = T;
  RowSinks o;
  o.codes = Xq;
  o.scale = s_a;
  o.copy = X;
  o.u = Xu;
  o.sum_u = sum_xu;
  return from_cuda(counted(launch_quant_rows(src, B * (params->K + T), d, o, s)));
}

}  // extern "C"

// ---------------------------------------------------------------------------
// Selector without a caller-provided workspace.
//
// Some callers cannot allocate device memory at the point where they run the
// selector: code inside a fixed memory budget set up once at start-up, plugins
// called from a runtime that owns the allocator, or hosts that must not
// allocate while other work is in flight. p4q_select_noalloc gives them the
// same selection with its scratch in the fixed array below. That array is
// part of this library's device image, so every GPU that loads the library
// reserves its bytes until the process exits.
// ---------------------------------------------------------------------------
namespace {

constexpr size_t kNoAllocScratchBytes = P4Q_NOALLOC_SCRATCH_BYTES;
static __device__ __align__(256) unsigned char g_select_scratch[kNoAllocScratchBytes];

// Device address of g_select_scratch in the current context. Host code cannot
// use the symbol itself: in host code it names a host-side placeholder, not
// device memory. The address is looked up on every call (a host-side table
// read once the module is loaded), so it stays right after cudaDeviceReset or
// under another context of the same device.
p4q_status scratch_address(void** out) {
  void* ptr = nullptr;
  if (cudaGetSymbolAddress(&ptr, g_select_scratch) != cudaSuccess || ptr == nullptr) return P4Q_ERR_CUDA;
  *out = ptr;
  return P4Q_OK;
}

}  // namespace

extern "C" p4q_status p4q_select_noalloc(const uint16_t* V, int B, int N, int d, const uint16_t* Q, int J,
                                         const float* A_cls, const p4q_select_params* params, int32_t* idx,
                                         p4q_stream_t stream) {
  p4q_status st = check_select_args(V, B, N, d, J, params, idx);
  if (st != P4Q_OK) return st;
  const bool have_q = (Q != nullptr && J > 0);
  const int Jeff = have_q ? J : 0;
  // Every region of the scratch is written before it is read on each call, so
  // nothing needs clearing between calls.
  const int r0 = select_r0(*params, have_q, A_cls != nullptr);
  const int kd = params->K - r0;
  if (select_workspace_layout(B, N, d, Jeff, r0, select_candidates(N, r0, kd), select_gram_mode(N, kd), nullptr,
                              nullptr) > kNoAllocScratchBytes)
    return P4Q_ERR_WORKSPACE_TOO_SMALL;
  if ((st = check_device()) != P4Q_OK) return st;
  void* ws = nullptr;
  if ((st = scratch_address(&ws)) != P4Q_OK) return st;
  // serial order on `stream`: the call creates no stream or event either
  return run_select(V, B, N, d, Q, J, A_cls, params, idx, ws, kNoAllocScratchBytes,
                    reinterpret_cast<cudaStream_t>(stream), false);
}

