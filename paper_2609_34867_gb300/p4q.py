"""Thin Python binding of libp4q.so (include/p4q.h), argument marshalling only.

Each function has the name of the C entry point it calls and passes torch
tensors as raw device pointers plus the current CUDA stream; every step of the
work runs in the library's sm_103a kernels. A missing library raises: there is
no fallback path.
"""
from __future__ import annotations

import ctypes
import os

import torch

from . import build as _build

P4Q_OK = 0
STATUS_NAMES = {0: "P4Q_OK", 1: "P4Q_ERR_INVALID_ARG", 2: "P4Q_ERR_UNSUPPORTED_SHAPE", 3: "P4Q_ERR_MISALIGNED",
                4: "P4Q_ERR_WORKSPACE_TOO_SMALL", 5: "P4Q_ERR_CUDA", 6: "P4Q_ERR_TIMEOUT", 7: "P4Q_ERR_NO_DEVICE"}


class P4QError(RuntimeError):
    def __init__(self, status: int, what: str):
        self.status = status
        super().__init__(f"{what}: {STATUS_NAMES.get(status, status)} ({p4q_status_string(status)})")


class SelectParams(ctypes.Structure):
    _fields_ = [("K", ctypes.c_int32), ("alpha_permille", ctypes.c_int32), ("beta_permille", ctypes.c_int32)]


_lib = None


def lib() -> ctypes.CDLL:
    """The loaded libp4q.so (raises if it has not been built)."""
    global _lib
    if _lib is None:
        if not os.path.exists(_build.LIB):
            raise RuntimeError(f"{_build.LIB} is missing: run __graft_entry__.build() first")
        L = ctypes.CDLL(_build.LIB)
        P, I, S = ctypes.c_void_p, ctypes.c_int, ctypes.c_size_t
        st = ctypes.c_int
        L.p4q_status_string.argtypes = [st]
        L.p4q_status_string.restype = ctypes.c_char_p
        L.p4q_launch_count.argtypes = []
        L.p4q_launch_count.restype = ctypes.c_uint64
        L.p4q_set_gemm_variant.argtypes = [I]
        L.p4q_set_gemm_variant.restype = st
        L.p4q_cls_saliency.argtypes = [P, P, P, I, I, I, I, I, P, P]
        L.p4q_cls_saliency.restype = st
        L.p4q_swiglu_quant_expanded.argtypes = [P, I, P, I, I, I, P, P, P, P, P]
        L.p4q_swiglu_quant_expanded.restype = st
        L.p4q_rmsnorm_quant_expanded.argtypes = [P, I, P, ctypes.c_float, I, I, P, P, P, P, P]
        L.p4q_rmsnorm_quant_expanded.restype = st
        L.p4q_causal_attention.argtypes = [P, I, P, I, P, I, I, I, I, I, I, P, I, P]
        L.p4q_causal_attention.restype = st
        L.p4q_block_mse_workspace_bytes.argtypes = [I]
        L.p4q_block_mse_workspace_bytes.restype = S
        L.p4q_block_mse.argtypes = [P, I, P, I, P, I, I, P, P, P, S, P]
        L.p4q_block_mse.restype = st
        L.p4q_topk_replacement.argtypes = [P, P, I, I, I, P, P, P]
        L.p4q_topk_replacement.restype = st
        L.p4q_device_status.argtypes = [P]
        L.p4q_device_status.restype = st
        L.p4q_test_wait_timeout.argtypes = [ctypes.c_uint32, P]
        L.p4q_test_wait_timeout.restype = st
        L.p4q_peak_probe.argtypes = [I, I, P, ctypes.POINTER(ctypes.c_double), P]
        L.p4q_peak_probe.restype = st
        L.p4q_quant_act.argtypes = [P, I, I, P, P, P]
        L.p4q_quant_act.restype = st
        L.p4q_quant_act_ld.argtypes = [P, I, I, I, P, P, P]
        L.p4q_quant_act_ld.restype = st
        L.p4q_quant_act_expanded.argtypes = [P, I, I, I, P, P, P, P, P]
        L.p4q_quant_act_expanded.restype = st
        L.p4q_select_gather_quant_expanded.argtypes = [P, I, I, I, P, I, P, P, I, ctypes.POINTER(SelectParams), P,
                                                       P, P, P, P, P, P, S, P]
        L.p4q_select_gather_quant_expanded.restype = st
        L.p4q_quant_weight.argtypes = [P, I, I, P, P, P]
        L.p4q_quant_weight.restype = st
        L.p4q_w4a4_linear.argtypes = [P, P, I, I, P, P, I, P, P]
        L.p4q_w4a4_linear.restype = st
        L.p4q_w4a4_gemm_s32.argtypes = [P, I, I, P, I, P, P]
        L.p4q_w4a4_gemm_s32.restype = st
        L.p4q_w4a4_linear_workspace_bytes.argtypes = [I, I, I]
        L.p4q_w4a4_linear_workspace_bytes.restype = S
        L.p4q_w4a4_linear_ws.argtypes = [P, P, I, I, P, P, I, P, P, S, P]
        L.p4q_w4a4_linear_ws.restype = st
        L.p4q_w4a4_gemm_s32_ws.argtypes = [P, I, I, P, I, P, P, S, P]
        L.p4q_w4a4_gemm_s32_ws.restype = st
        L.p4q_expand_codes.argtypes = [P, I, I, P, P, P]
        L.p4q_expand_codes.restype = st
        L.p4q_w4a4_linear_expanded.argtypes = [P, P, P, I, I, P, P, P, I, P, P]
        L.p4q_w4a4_linear_expanded.restype = st
        L.p4q_w4a4_linear_expanded_rowmax.argtypes = [P, P, P, I, I, P, P, P, I, P, I, P, P, P, P]
        L.p4q_w4a4_linear_expanded_rowmax.restype = st
        L.p4q_quant_act_expanded_rowmax.argtypes = [P, I, I, I, P, P, P, P, P, P, P, P]
        L.p4q_quant_act_expanded_rowmax.restype = st
        L.p4q_select_workspace_bytes.argtypes = [I, I, I, I, ctypes.POINTER(SelectParams)]
        L.p4q_select_workspace_bytes.restype = S
        L.p4q_select.argtypes = [P, I, I, I, P, I, P, ctypes.POINTER(SelectParams), P, P, S, P]
        L.p4q_select.restype = st
        L.p4q_select_gather_quant.argtypes = [P, I, I, I, P, I, P, P, I, ctypes.POINTER(SelectParams), P, P, P,
                                              P, P, S, P]
        L.p4q_select_gather_quant.restype = st
        _lib = L
    return _lib


def _ptr(t):
    return None if t is None else ctypes.c_void_p(t.data_ptr())


def _stream(stream):
    if stream is None:
        stream = torch.cuda.current_stream()
    return ctypes.c_void_p(stream.cuda_stream)


def _check(status: int, what: str):
    if status != P4Q_OK:
        raise P4QError(status, what)


def _need(t, dtype, ndim, name):
    if not isinstance(t, torch.Tensor) or t.dtype != dtype or t.dim() != ndim or not t.is_contiguous():
        raise TypeError(f"{name}: expected a contiguous {dtype} tensor with {ndim} dims")
    if not t.is_cuda:
        raise TypeError(f"{name}: expected a CUDA tensor")


def p4q_status_string(status: int) -> str:
    return lib().p4q_status_string(int(status)).decode()


def p4q_launch_count() -> int:
    """Kernels launched by libp4q.so in this process so far."""
    return int(lib().p4q_launch_count())


def p4q_set_gemm_variant(variant: int):
    """0 automatic, 1 single-CTA GEMM only, 2 CTA-pair GEMM whenever N >= 256,
    3 automatic with the expanded-operand path whenever a workspace is given."""
    _check(lib().p4q_set_gemm_variant(int(variant)), "p4q_set_gemm_variant")


def p4q_device_status(stream=None) -> int:
    return int(lib().p4q_device_status(_stream(stream)))


PEAK_KINDS = {"f8": 0, "s8": 1, "dp4a": 2}


def p4q_peak_probe(kind: str, iters: int, sink, stream=None) -> float:
    """Launches one throughput probe (f8: tcgen05 kind::f8f6f4 MMAs, s8:
    mma.sync m16n8k32 s8, dp4a) on `stream`; returns the operations it performs.
    sink: a CUDA int32 tensor of at least 8192 elements."""
    _need(sink, torch.int32, 1, "sink")
    if sink.numel() < 8192:
        raise ValueError("sink: at least 8192 elements")
    ops = ctypes.c_double(0.0)
    _check(lib().p4q_peak_probe(PEAK_KINDS[kind], iters, _ptr(sink), ctypes.byref(ops), _stream(stream)),
           "p4q_peak_probe")
    return ops.value


def p4q_quant_act(X, Xq, s_a, stream=None):
    """X [M, Kin] fp16 -> Xq [M, Kin/2] uint8 (packed INT4), s_a [M] fp32."""
    _need(X, torch.float16, 2, "X"); _need(Xq, torch.uint8, 2, "Xq"); _need(s_a, torch.float32, 1, "s_a")
    M, K = X.shape
    _check(lib().p4q_quant_act(_ptr(X), M, K, _ptr(Xq), _ptr(s_a), _stream(stream)), "p4q_quant_act")


def p4q_quant_act_ld(X, Xq, s_a, stream=None):
    """p4q_quant_act on a row-strided 2-D view X (unit column stride, rows
    X.stride(0) elements apart), e.g. a column block of a fused output."""
    if not isinstance(X, torch.Tensor) or X.dtype != torch.float16 or X.dim() != 2 or X.stride(1) != 1 or not X.is_cuda:
        raise TypeError("X: expected a CUDA fp16 2-D tensor with unit column stride")
    _need(Xq, torch.uint8, 2, "Xq"); _need(s_a, torch.float32, 1, "s_a")
    M, K = X.shape
    _check(lib().p4q_quant_act_ld(_ptr(X), X.stride(0), M, K, _ptr(Xq), _ptr(s_a), _stream(stream)),
           "p4q_quant_act_ld")


def p4q_quant_act_expanded(X, Xq, s_a, Xu, sum_xu, stream=None):
    """p4q_quant_act_ld plus the expanded codes (see p4q_expand_codes)."""
    if not isinstance(X, torch.Tensor) or X.dtype != torch.float16 or X.dim() != 2 or X.stride(1) != 1 or not X.is_cuda:
        raise TypeError("X: expected a CUDA fp16 2-D tensor with unit column stride")
    _need(Xq, torch.uint8, 2, "Xq"); _need(s_a, torch.float32, 1, "s_a")
    _need(Xu, torch.uint8, 2, "Xu"); _need(sum_xu, torch.int32, 1, "sum_xu")
    M, K = X.shape
    _check(lib().p4q_quant_act_expanded(_ptr(X), X.stride(0), M, K, _ptr(Xq), _ptr(s_a), _ptr(Xu), _ptr(sum_xu),
                                        _stream(stream)), "p4q_quant_act_expanded")


def p4q_swiglu_quant_expanded(gate, up, Xq, s_a, Xu=None, sum_xu=None, stream=None):
    """Codes of silu(gate) * up per row (gate, up: [M, Kin] fp16 views with unit
    column stride, e.g. column blocks of a fused gate|up output); Xu / sum_xu
    optional (both or neither)."""
    for t, name in ((gate, "gate"), (up, "up")):
        if not isinstance(t, torch.Tensor) or t.dtype != torch.float16 or t.dim() != 2 or t.stride(1) != 1 or \
                not t.is_cuda:
            raise TypeError(f"{name}: expected a CUDA fp16 2-D tensor with unit column stride")
    _need(Xq, torch.uint8, 2, "Xq"); _need(s_a, torch.float32, 1, "s_a")
    if Xu is not None:
        _need(Xu, torch.uint8, 2, "Xu"); _need(sum_xu, torch.int32, 1, "sum_xu")
    M, K = gate.shape
    _check(lib().p4q_swiglu_quant_expanded(_ptr(gate), gate.stride(0), _ptr(up), up.stride(0), M, K, _ptr(Xq),
                                           _ptr(s_a), _ptr(Xu), _ptr(sum_xu), _stream(stream)),
           "p4q_swiglu_quant_expanded")


def p4q_rmsnorm_quant_expanded(X, w, eps, Xq, s_a, Xu=None, sum_xu=None, stream=None):
    """Codes of the RMSNorm of each row of X ([M, Kin] fp16 view with unit
    column stride) with gain w ([Kin] fp16) and epsilon eps; Xu / sum_xu
    optional (both or neither)."""
    if not isinstance(X, torch.Tensor) or X.dtype != torch.float16 or X.dim() != 2 or X.stride(1) != 1 or \
            not X.is_cuda:
        raise TypeError("X: expected a CUDA fp16 2-D tensor with unit column stride")
    _need(w, torch.float16, 1, "w"); _need(Xq, torch.uint8, 2, "Xq"); _need(s_a, torch.float32, 1, "s_a")
    if Xu is not None:
        _need(Xu, torch.uint8, 2, "Xu"); _need(sum_xu, torch.int32, 1, "sum_xu")
    M, K = X.shape
    if w.shape[0] != K:
        raise ValueError(f"w has {w.shape[0]} values, X rows have {K}")
    _check(lib().p4q_rmsnorm_quant_expanded(_ptr(X), X.stride(0), _ptr(w), float(eps), M, K, _ptr(Xq), _ptr(s_a),
                                            _ptr(Xu), _ptr(sum_xu), _stream(stream)),
           "p4q_rmsnorm_quant_expanded")


def p4q_causal_attention(q, k, v, o, B, m, H, Hkv, stream=None):
    """Causal attention per sample and head on fp16 rows (head dim 128): q, o
    [B*m, >= H*128], k, v [B*m, >= Hkv*128], 2-D views with unit column stride
    (e.g. column blocks of a fused projection output)."""
    for t, name in ((q, "q"), (k, "k"), (v, "v"), (o, "o")):
        if not isinstance(t, torch.Tensor) or t.dtype != torch.float16 or t.dim() != 2 or t.stride(1) != 1 or \
                not t.is_cuda or t.shape[0] != B * m:
            raise TypeError(f"{name}: expected a CUDA fp16 2-D tensor of B*m rows with unit column stride")
    _check(lib().p4q_causal_attention(_ptr(q), q.stride(0), _ptr(k), k.stride(0), _ptr(v), v.stride(0), B, m, H,
                                      Hkv, 128, _ptr(o), o.stride(0), _stream(stream)), "p4q_causal_attention")


def p4q_block_mse_workspace_bytes(B):
    return int(lib().p4q_block_mse_workspace_bytes(int(B)))


def p4q_block_mse(Yq, Yf, offsets, e, L, ws, stream=None):
    """Eq. 5's block objective: Yq, Yf [rows, d] fp16 2-D views with unit column
    stride; offsets a host sequence of B + 1 row offsets; e [B], L [1] fp32;
    ws a uint8 device buffer of p4q_block_mse_workspace_bytes(B) bytes."""
    for t, name in ((Yq, "Yq"), (Yf, "Yf")):
        if not isinstance(t, torch.Tensor) or t.dtype != torch.float16 or t.dim() != 2 or t.stride(1) != 1 or \
                not t.is_cuda:
            raise TypeError(f"{name}: expected a CUDA fp16 2-D tensor with unit column stride")
    if Yq.shape != Yf.shape:
        raise ValueError("Yq and Yf differ in shape")
    off = (ctypes.c_int32 * len(offsets))(*[int(x) for x in offsets])
    B = len(offsets) - 1
    if B >= 1 and int(offsets[-1]) > Yq.shape[0]:
        raise ValueError("offsets run past the rows of Yq")
    _need(e, torch.float32, 1, "e"); _need(L, torch.float32, 1, "L"); _need(ws, torch.uint8, 1, "ws")
    _check(lib().p4q_block_mse(_ptr(Yq), Yq.stride(0), _ptr(Yf), Yf.stride(0), off, B, Yq.shape[1], _ptr(e), _ptr(L),
                               _ptr(ws), ws.numel(), _stream(stream)), "p4q_block_mse")


def p4q_topk_replacement(s_ref, s_alt, K, inter, rho, stream=None):
    """Eq. 9's replacement ratio: s_ref, s_alt [B, N] fp32 -> inter [B] int32, rho [B] fp32."""
    _need(s_ref, torch.float32, 2, "s_ref"); _need(s_alt, torch.float32, 2, "s_alt")
    _need(inter, torch.int32, 1, "inter"); _need(rho, torch.float32, 1, "rho")
    if s_ref.shape != s_alt.shape:
        raise ValueError("score rows differ in shape")
    B, N = s_ref.shape
    _check(lib().p4q_topk_replacement(_ptr(s_ref), _ptr(s_alt), B, N, int(K), _ptr(inter), _ptr(rho),
                                      _stream(stream)), "p4q_topk_replacement")


def p4q_quant_weight(W, Wq, s_w, stream=None):
    """W [N, Kin] fp16 -> Wq [N, Kin/2] uint8, s_w [N] fp32 (one scale per output channel)."""
    _need(W, torch.float16, 2, "W"); _need(Wq, torch.uint8, 2, "Wq"); _need(s_w, torch.float32, 1, "s_w")
    N, K = W.shape
    _check(lib().p4q_quant_weight(_ptr(W), N, K, _ptr(Wq), _ptr(s_w), _stream(stream)), "p4q_quant_weight")


def p4q_w4a4_linear(Xq, s_a, Wq, s_w, Y, stream=None):
    """Y [M, N] fp16 = dequant(Xq Wq^T) with per-token s_a and per-channel s_w."""
    _need(Xq, torch.uint8, 2, "Xq"); _need(Wq, torch.uint8, 2, "Wq"); _need(Y, torch.float16, 2, "Y")
    M, K = Xq.shape[0], Xq.shape[1] * 2
    N = Wq.shape[0]
    _check(lib().p4q_w4a4_linear(_ptr(Xq), _ptr(s_a), M, K, _ptr(Wq), _ptr(s_w), N, _ptr(Y), _stream(stream)),
           "p4q_w4a4_linear")


def p4q_w4a4_gemm_s32(Xq, Wq, acc, stream=None):
    """acc [M, N] int32 = exact integer product of the packed INT4 codes."""
    _need(Xq, torch.uint8, 2, "Xq"); _need(Wq, torch.uint8, 2, "Wq"); _need(acc, torch.int32, 2, "acc")
    M, K = Xq.shape[0], Xq.shape[1] * 2
    N = Wq.shape[0]
    _check(lib().p4q_w4a4_gemm_s32(_ptr(Xq), M, K, _ptr(Wq), N, _ptr(acc), _stream(stream)), "p4q_w4a4_gemm_s32")


def p4q_select_workspace_bytes(B: int, N: int, d: int, J: int, K: int, alpha_permille: int = 300,
                               beta_permille: int = 200) -> int:
    p = SelectParams(K, alpha_permille, beta_permille)
    return int(lib().p4q_select_workspace_bytes(B, N, d, J, ctypes.byref(p)))


def p4q_select(V, Q, A_cls, K, idx, ws, alpha_permille=300, beta_permille=200, stream=None):
    """V [B, N, d] fp16, Q [B, J, d] fp16 or None, A_cls [B, N] fp32 or None -> idx [B, K] int32."""
    _need(V, torch.float16, 3, "V"); _need(idx, torch.int32, 2, "idx"); _need(ws, torch.uint8, 1, "ws")
    B, N, d = V.shape
    J = 0 if Q is None else Q.shape[1]
    p = SelectParams(K, alpha_permille, beta_permille)
    _check(lib().p4q_select(_ptr(V), B, N, d, _ptr(Q), J, _ptr(A_cls), ctypes.byref(p), _ptr(idx), _ptr(ws),
                            ws.numel(), _stream(stream)), "p4q_select")


def p4q_select_gather_quant(V, Q, A_cls, text, K, idx, X, Xq, s_a, ws, alpha_permille=300, beta_permille=200,
                            stream=None):
    """Selector, gather of [kept V rows; text rows] into X [B, K+T, d] fp16, and its INT4 quantization."""
    _need(V, torch.float16, 3, "V"); _need(idx, torch.int32, 2, "idx"); _need(ws, torch.uint8, 1, "ws")
    _need(X, torch.float16, 3, "X"); _need(Xq, torch.uint8, 2, "Xq"); _need(s_a, torch.float32, 1, "s_a")
    B, N, d = V.shape
    J = 0 if Q is None else Q.shape[1]
    T = 0 if text is None else text.shape[1]
    p = SelectParams(K, alpha_permille, beta_permille)
    _check(lib().p4q_select_gather_quant(_ptr(V), B, N, d, _ptr(Q), J, _ptr(A_cls), _ptr(text), T,
                                         ctypes.byref(p), _ptr(idx), _ptr(X), _ptr(Xq), _ptr(s_a), _ptr(ws),
                                         ws.numel(), _stream(stream)), "p4q_select_gather_quant")


def p4q_select_gather_quant_expanded(V, Q, A_cls, text, K, idx, X, Xq, s_a, Xu, sum_xu, ws, alpha_permille=300,
                                     beta_permille=200, stream=None):
    """p4q_select_gather_quant plus the pruned sequence's expanded codes (see p4q_expand_codes);
    Xq may be None (only the expanded codes are written)."""
    _need(V, torch.float16, 3, "V"); _need(idx, torch.int32, 2, "idx"); _need(ws, torch.uint8, 1, "ws")
    _need(X, torch.float16, 3, "X"); _need(s_a, torch.float32, 1, "s_a")
    if Xq is not None:
        _need(Xq, torch.uint8, 2, "Xq")
    _need(Xu, torch.uint8, 2, "Xu"); _need(sum_xu, torch.int32, 1, "sum_xu")
    B, N, d = V.shape
    J = 0 if Q is None else Q.shape[1]
    T = 0 if text is None else text.shape[1]
    p = SelectParams(K, alpha_permille, beta_permille)
    _check(lib().p4q_select_gather_quant_expanded(_ptr(V), B, N, d, _ptr(Q), J, _ptr(A_cls), _ptr(text), T,
                                                  ctypes.byref(p), _ptr(idx), _ptr(X), _ptr(Xq), _ptr(s_a), _ptr(Xu),
                                                  _ptr(sum_xu), _ptr(ws), ws.numel(), _stream(stream)),
           "p4q_select_gather_quant_expanded")


def p4q_cls_saliency(q_cls, k_cls, k, A_cls, stream=None):
    """A_cls [B, N] fp32 from the final-layer CLS query/key [B, C, H, dh] and
    patch keys [B, N, H, dh] (fp16, contiguous)."""
    _need(q_cls, torch.float16, 4, "q_cls"); _need(k_cls, torch.float16, 4, "k_cls")
    _need(k, torch.float16, 4, "k"); _need(A_cls, torch.float32, 2, "A_cls")
    B, C, H, dh = q_cls.shape
    N = k.shape[1]
    _check(lib().p4q_cls_saliency(_ptr(q_cls), _ptr(k_cls), _ptr(k), B, N, C, H, dh, _ptr(A_cls), _stream(stream)),
           "p4q_cls_saliency")


def cls_saliency(q_cls, k_cls, k, stream=None):
    """Allocating wrapper of p4q_cls_saliency."""
    A = torch.empty((q_cls.shape[0], k.shape[1]), dtype=torch.float32, device=k.device)
    p4q_cls_saliency(q_cls, k_cls, k, A, stream)
    return A


# ---------------------------------------------------------------- helpers
def quant_act(X, stream=None):
    """Allocating wrapper of p4q_quant_act: returns (Xq, s_a)."""
    M, K = X.shape
    Xq = torch.empty((M, K // 2), dtype=torch.uint8, device=X.device)
    s = torch.empty((M,), dtype=torch.float32, device=X.device)
    p4q_quant_act(X, Xq, s, stream)
    return Xq, s


def quant_weight(W, stream=None):
    N, K = W.shape
    Wq = torch.empty((N, K // 2), dtype=torch.uint8, device=W.device)
    s = torch.empty((N,), dtype=torch.float32, device=W.device)
    p4q_quant_weight(W, Wq, s, stream)
    return Wq, s


def w4a4_linear(Xq, s_a, Wq, s_w, stream=None):
    Y = torch.empty((Xq.shape[0], Wq.shape[0]), dtype=torch.float16, device=Xq.device)
    p4q_w4a4_linear(Xq, s_a, Wq, s_w, Y, stream)
    return Y


def linear_workspace(M, N, K, device):
    """A device workspace large enough for p4q_w4a4_linear_ws on M x N x K."""
    n = int(lib().p4q_w4a4_linear_workspace_bytes(int(M), int(N), int(K)))
    if n == 0:
        raise P4QError(1, "p4q_w4a4_linear_workspace_bytes")
    return torch.empty((n,), dtype=torch.uint8, device=device)


def p4q_w4a4_linear_ws(Xq, s_a, Wq, s_w, Y, ws, stream=None):
    """p4q_w4a4_linear with a caller workspace (None: no workspace)."""
    _need(Xq, torch.uint8, 2, "Xq"); _need(Wq, torch.uint8, 2, "Wq"); _need(Y, torch.float16, 2, "Y")
    M, K = Xq.shape[0], Xq.shape[1] * 2
    N = Wq.shape[0]
    wp, wn = (None, 0) if ws is None else (_ptr(ws), ws.numel() * ws.element_size())
    _check(lib().p4q_w4a4_linear_ws(_ptr(Xq), _ptr(s_a), M, K, _ptr(Wq), _ptr(s_w), N, _ptr(Y), wp, wn,
                                    _stream(stream)), "p4q_w4a4_linear_ws")


def w4a4_gemm_s32_ws(Xq, Wq, ws, stream=None):
    """Allocating wrapper of p4q_w4a4_gemm_s32_ws: returns the int32 accumulators."""
    M, K = Xq.shape[0], Xq.shape[1] * 2
    N = Wq.shape[0]
    acc = torch.empty((M, N), dtype=torch.int32, device=Xq.device)
    wp, wn = (None, 0) if ws is None else (_ptr(ws), ws.numel() * ws.element_size())
    _check(lib().p4q_w4a4_gemm_s32_ws(_ptr(Xq), M, K, _ptr(Wq), N, _ptr(acc), wp, wn, _stream(stream)),
           "p4q_w4a4_gemm_s32_ws")
    return acc


def p4q_expand_codes(q, u, sum_u, stream=None):
    """Packed codes q [rows, K/2] uint8 -> u [rows, K] uint8 (u = v + 8), sum_u [rows] int32."""
    _need(q, torch.uint8, 2, "q"); _need(u, torch.uint8, 2, "u"); _need(sum_u, torch.int32, 1, "sum_u")
    rows, K = q.shape[0], q.shape[1] * 2
    _check(lib().p4q_expand_codes(_ptr(q), rows, K, _ptr(u), _ptr(sum_u), _stream(stream)), "p4q_expand_codes")


def expand_codes(q, stream=None):
    """Allocating wrapper of p4q_expand_codes: returns (u, sum_u)."""
    u = torch.empty((q.shape[0], q.shape[1] * 2), dtype=torch.uint8, device=q.device)
    s = torch.empty((q.shape[0],), dtype=torch.int32, device=q.device)
    p4q_expand_codes(q, u, s, stream)
    return u, s


def p4q_w4a4_linear_expanded(Xu, sum_xu, s_a, Wu, sum_wu, s_w, Y, stream=None):
    """Y [M, N] fp16 from expanded operands (see p4q_expand_codes)."""
    _need(Xu, torch.uint8, 2, "Xu"); _need(Wu, torch.uint8, 2, "Wu"); _need(Y, torch.float16, 2, "Y")
    M, K = Xu.shape
    N = Wu.shape[0]
    _check(lib().p4q_w4a4_linear_expanded(_ptr(Xu), _ptr(sum_xu), _ptr(s_a), M, K, _ptr(Wu), _ptr(sum_wu), _ptr(s_w),
                                          N, _ptr(Y), _stream(stream)), "p4q_w4a4_linear_expanded")


def _host_ints(vals):
    return (ctypes.c_int * len(vals))(*vals)


def _host_ptrs(ts):
    return (ctypes.c_void_p * len(ts))(*[(_ptr(t) if t is not None else None) for t in ts])


def p4q_w4a4_linear_expanded_rowmax(Xu, sum_xu, s_a, Wu, sum_wu, s_w, Y, blocks, rowmax, stream=None):
    """p4q_w4a4_linear_expanded plus each row's |Y| abs-max (fp16 bits) over
    the column blocks [(col0, ncols), ...] (at most two) into rowmax [nblk, M]."""
    _need(Xu, torch.uint8, 2, "Xu"); _need(Wu, torch.uint8, 2, "Wu"); _need(Y, torch.float16, 2, "Y")
    _need(rowmax, torch.int32, 2, "rowmax")
    M, K = Xu.shape
    N = Wu.shape[0]
    c0, nc = _host_ints([b[0] for b in blocks]), _host_ints([b[1] for b in blocks])
    _check(lib().p4q_w4a4_linear_expanded_rowmax(_ptr(Xu), _ptr(sum_xu), _ptr(s_a), M, K, _ptr(Wu), _ptr(sum_wu),
                                                 _ptr(s_w), N, _ptr(Y), len(blocks), c0, nc, _ptr(rowmax),
                                                 _stream(stream)), "p4q_w4a4_linear_expanded_rowmax")


def p4q_quant_act_expanded_rowmax(Y, blocks, rowmax, Xq, s_a, Xu, sum_xu, stream=None):
    """p4q_quant_act_expanded of the column blocks [(col0, ncols), ...] of Y with
    the row abs-max given; Xq, s_a, Xu, sum_xu: one tensor per block (Xq
    entries may be None)."""
    if not isinstance(Y, torch.Tensor) or Y.dtype != torch.float16 or Y.dim() != 2 or Y.stride(1) != 1 or not Y.is_cuda:
        raise TypeError("Y: expected a CUDA fp16 2-D tensor with unit column stride")
    _need(rowmax, torch.int32, 2, "rowmax")
    for b in range(len(blocks)):
        if Xq is not None and Xq[b] is not None:
            _need(Xq[b], torch.uint8, 2, "Xq")
        _need(s_a[b], torch.float32, 1, "s_a"); _need(Xu[b], torch.uint8, 2, "Xu")
        _need(sum_xu[b], torch.int32, 1, "sum_xu")
    c0, nc = _host_ints([b[0] for b in blocks]), _host_ints([b[1] for b in blocks])
    _check(lib().p4q_quant_act_expanded_rowmax(_ptr(Y), Y.stride(0), Y.shape[0], len(blocks), c0, nc, _ptr(rowmax),
                                               _host_ptrs(Xq) if Xq is not None else None, _host_ptrs(s_a),
                                               _host_ptrs(Xu), _host_ptrs(sum_xu),
                                               _stream(stream)), "p4q_quant_act_expanded_rowmax")


def w4a4_gemm_s32(Xq, Wq, stream=None):
    acc = torch.empty((Xq.shape[0], Wq.shape[0]), dtype=torch.int32, device=Xq.device)
    p4q_w4a4_gemm_s32(Xq, Wq, acc, stream)
    return acc


def select_workspace(B, N, d, J, K, device, alpha_permille=300, beta_permille=200):
    n = p4q_select_workspace_bytes(B, N, d, J, K, alpha_permille, beta_permille)
    if n == 0:
        raise P4QError(1, "p4q_select_workspace_bytes")
    return torch.empty((n,), dtype=torch.uint8, device=device)


def select(V, Q, A_cls, K, ws=None, alpha_permille=300, beta_permille=200, stream=None):
    B, N, d = V.shape
    J = 0 if Q is None else Q.shape[1]
    if ws is None:
        ws = select_workspace(B, N, d, J, K, V.device, alpha_permille, beta_permille)
    idx = torch.empty((B, K), dtype=torch.int32, device=V.device)
    p4q_select(V, Q, A_cls, K, idx, ws, alpha_permille, beta_permille, stream)
    return idx


def select_gather_quant(V, Q, A_cls, text, K, ws=None, alpha_permille=300, beta_permille=200, stream=None):
    B, N, d = V.shape
    J = 0 if Q is None else Q.shape[1]
    T = 0 if text is None else text.shape[1]
    if ws is None:
        ws = select_workspace(B, N, d, J, K, V.device, alpha_permille, beta_permille)
    idx = torch.empty((B, K), dtype=torch.int32, device=V.device)
    X = torch.empty((B, K + T, d), dtype=torch.float16, device=V.device)
    Xq = torch.empty((B * (K + T), d // 2), dtype=torch.uint8, device=V.device)
    s_a = torch.empty((B * (K + T),), dtype=torch.float32, device=V.device)
    p4q_select_gather_quant(V, Q, A_cls, text, K, idx, X, Xq, s_a, ws, alpha_permille, beta_permille, stream)
    return idx, X, Xq, s_a
