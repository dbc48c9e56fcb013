"""CPU oracle for the P4Q pruned W4A4 hot path (test infrastructure only).

Only the tests, ``__graft_entry__.smoke()`` and the CPU-baseline leg of
``bench.py`` may import this package. It is a thin ctypes wrapper around
``p4q_oracle.c`` (plain C11, compiled with gcc) and shares no code with the
CUDA library. Every function here marshals numpy arrays; the arithmetic lives
in the C file, which cites the paper passage each step follows (Sec. 3.2,
Eq. 4 for the selector and the CLS saliency; App. A and App. B.3 for the
W4A4 quantizer).

fp16 inputs are widened to fp32 with numpy before the call; that conversion is
exact, so the oracle sees the same values as the GPU path.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "p4q_oracle.c")
_LIB = os.path.join(_HERE, "libp4q_oracle.so")
_lock = threading.Lock()
_lib = None

OK, BAD_ARG, OVERFLOW = 0, 1, 2


def build(force: bool = False) -> str:
    """Compile the oracle with gcc (no fast-math, no FMA contraction)."""
    if force or not os.path.exists(_LIB) or os.path.getmtime(_LIB) < os.path.getmtime(_SRC):
        tmp = _LIB + f".tmp{os.getpid()}"
        cmd = ["gcc", "-std=c11", "-O2", "-ffp-contract=off", "-fno-fast-math", "-fopenmp",
               "-fPIC", "-shared", "-Wall", "-o", tmp, _SRC, "-lm"]
        subprocess.run(cmd, check=True)
        os.replace(tmp, _LIB)
    return _LIB


def _load():
    global _lib
    with _lock:
        if _lib is None:
            build()
            lib = ctypes.CDLL(_LIB)
            P = ctypes.c_void_p
            i64, i32, f32 = ctypes.c_int64, ctypes.c_int, ctypes.c_float
            lib.oracle_set_threads.argtypes = [i32]
            lib.oracle_set_threads.restype = i32
            lib.q4_quantize_rows.argtypes = [P, i64, i64, P, P]
            lib.q4_quantize_rows.restype = i32
            lib.q4_cosine.argtypes = [P, P, i64]
            lib.q4_cosine.restype = f32
            lib.p4q_budget.argtypes = [i32, i32, i32, i32, i32, P, P, P]
            lib.p4q_budget.restype = None
            lib.p4q_select_one.argtypes = [P, i32, i32, P, i32, P, i32, i32, i32, P, P, P]
            lib.p4q_select_one.restype = i32
            lib.p4q_select_batch.argtypes = [P, i32, i32, i32, P, i32, P, i32, i32, i32, P]
            lib.p4q_select_batch.restype = i32
            lib.w4a4_gemm_s32.argtypes = [P, P, i64, i64, i64, P]
            lib.w4a4_gemm_s32.restype = i32
            lib.w4a4_linear.argtypes = [P, P, P, P, i64, i64, i64, P]
            lib.w4a4_linear.restype = i32
            lib.p4q_gather.argtypes = [P, i32, i32, i32, P, i32, P, i32, P]
            lib.p4q_gather.restype = i32
            lib.p4q_cls_saliency.argtypes = [P, P, P, i32, i32, i32, i32, i32, P]
            lib.p4q_cls_saliency.restype = i32
            lib.p4q_swiglu_quantize_rows.argtypes = [P, P, i64, i64, P, P]
            lib.p4q_swiglu_quantize_rows.restype = i32
            lib.p4q_causal_attention.argtypes = [P, P, P, i32, i32, i32, i32, i32, P]
            lib.p4q_causal_attention.restype = i32
            lib.p4q_block_mse.argtypes = [P, P, P, i32, i32, P, P]
            lib.p4q_block_mse.restype = i32
            lib.p4q_topk_replacement.argtypes = [P, P, i32, i32, i32, P, P]
            lib.p4q_topk_replacement.restype = i32
            lib.oracle_sumsq32.argtypes = [P, i64]
            lib.oracle_sumsq32.restype = f32
            lib.p4q_rmsnorm_rows.argtypes = [P, P, f32, i64, i64, P]
            lib.p4q_rmsnorm_rows.restype = i32
            lib.p4q_rmsnorm_quantize_rows.argtypes = [P, P, f32, i64, i64, P, P]
            lib.p4q_rmsnorm_quantize_rows.restype = i32
            _lib = lib
    return _lib


def _f32(x):
    return np.ascontiguousarray(np.asarray(x).astype(np.float32, copy=False))


def _ptr(a):
    return None if a is None else a.ctypes.data


def set_threads(n: int) -> int:
    """Set the OpenMP thread count (n <= 0 keeps the default); returns the count in use."""
    return int(_load().oracle_set_threads(int(n)))


def quantize_rows(x):
    """Per-row symmetric 4-bit RTN quantizer. x: [rows, cols] (fp16 or fp32).

    Returns (codes int8 [rows, cols] in [-8, 7], scale float32 [rows]).
    """
    x = _f32(x)
    if x.ndim == 1:
        x = x[None]
    rows, cols = x.shape
    codes = np.empty((rows, cols), np.int8)
    scale = np.empty((rows,), np.float32)
    rc = _load().q4_quantize_rows(_ptr(x), rows, cols, _ptr(codes), _ptr(scale))
    if rc != OK:
        raise ValueError(f"oracle quantize_rows failed ({rc})")
    return codes, scale


def cosine(ca, cb) -> np.float32:
    """CosSim of two fake-quantized vectors, from their int8 codes."""
    ca = np.ascontiguousarray(ca, np.int8)
    cb = np.ascontiguousarray(cb, np.int8)
    assert ca.shape == cb.shape and ca.ndim == 1
    return np.float32(_load().q4_cosine(_ptr(ca), _ptr(cb), ca.shape[0]))


def budget(K: int, alpha_pm: int = 300, beta_pm: int = 200, have_q: bool = True, have_a: bool = True):
    """(K_q, K_s, K_d) of the budget split."""
    q, s, d = ctypes.c_int(), ctypes.c_int(), ctypes.c_int()
    _load().p4q_budget(int(K), int(alpha_pm), int(beta_pm), int(have_q), int(have_a),
                       ctypes.byref(q), ctypes.byref(s), ctypes.byref(d))
    return q.value, s.value, d.value


def select_one(V, K: int, Q=None, A=None, alpha_pm: int = 300, beta_pm: int = 200):
    """One image. V: [N, d]; Q: [J, d] or None; A: [N] or None.

    Returns (idx ascending [K], order [K] in pick order, stage [K]) where stage
    is 1 + concept index for query picks, -1 for saliency, -2 for diversity.
    """
    V = _f32(V)
    N, d = V.shape
    Qa = None if Q is None else _f32(Q)
    J = 0 if Qa is None else Qa.shape[0]
    Aa = None if A is None else _f32(A)
    idx = np.empty((K,), np.int32)
    order = np.empty((K,), np.int32)
    stage = np.empty((K,), np.int32)
    rc = _load().p4q_select_one(_ptr(V), N, d, _ptr(Qa), J, _ptr(Aa), int(K), int(alpha_pm),
                                int(beta_pm), _ptr(idx), _ptr(order), _ptr(stage))
    if rc != OK:
        raise ValueError(f"oracle select_one failed ({rc})")
    return idx, order, stage


def select_batch(V, K: int, Q=None, A=None, alpha_pm: int = 300, beta_pm: int = 200):
    """Batched selector. V: [B, N, d]; Q: [B, J, d] or None; A: [B, N] or None -> idx [B, K]."""
    V = _f32(V)
    B, N, d = V.shape
    Qa = None if Q is None else _f32(Q)
    J = 0 if Qa is None else Qa.shape[1]
    Aa = None if A is None else _f32(A)
    idx = np.empty((B, K), np.int32)
    rc = _load().p4q_select_batch(_ptr(V), B, N, d, _ptr(Qa), J, _ptr(Aa), int(K), int(alpha_pm),
                                  int(beta_pm), _ptr(idx))
    if rc != OK:
        raise ValueError(f"oracle select_batch failed ({rc})")
    return idx


def gemm_s32(a_codes, w_codes):
    """acc[m, n] = sum_k a[m, k] * w[n, k] on int8 codes; raises if it leaves int32."""
    a = np.ascontiguousarray(a_codes, np.int8)
    w = np.ascontiguousarray(w_codes, np.int8)
    M, K = a.shape
    N, K2 = w.shape
    assert K == K2
    acc = np.empty((M, N), np.int32)
    rc = _load().w4a4_gemm_s32(_ptr(a), _ptr(w), M, N, K, _ptr(acc))
    if rc != OK:
        raise OverflowError("oracle gemm accumulator left int32") if rc == OVERFLOW else ValueError(rc)
    return acc


def linear(a_codes, s_a, w_codes, s_w):
    """W4A4 linear in fp32: y = ((float)acc * s_a[m]) * s_w[n]."""
    a = np.ascontiguousarray(a_codes, np.int8)
    w = np.ascontiguousarray(w_codes, np.int8)
    sa = _f32(s_a).reshape(-1)
    sw = _f32(s_w).reshape(-1)
    M, K = a.shape
    N = w.shape[0]
    assert sa.shape[0] == M and sw.shape[0] == N and w.shape[1] == K
    y = np.empty((M, N), np.float32)
    rc = _load().w4a4_linear(_ptr(a), _ptr(sa), _ptr(w), _ptr(sw), M, N, K, _ptr(y))
    if rc != OK:
        raise ValueError(f"oracle linear failed ({rc})")
    return y


def gather(V, idx, text=None):
    """X = [V[b, idx[b]]; text[b]] per image, fp32. V: [B, N, d]; idx: [B, K]; text: [B, T, d]."""
    V = _f32(V)
    B, N, d = V.shape
    idx = np.ascontiguousarray(idx, np.int32)
    K = idx.shape[1]
    t = None if text is None else _f32(text)
    T = 0 if t is None else t.shape[1]
    X = np.empty((B, K + T, d), np.float32)
    rc = _load().p4q_gather(_ptr(V), B, N, d, _ptr(idx), K, _ptr(t), T, _ptr(X))
    if rc != OK:
        raise ValueError(f"oracle gather failed ({rc})")
    return X


def cls_saliency(q_cls, k_cls, k):
    """A_cls [B, N] (fp64) from the vision tower's final-layer attention (Sec. 3.2,
    Visual Saliency): per crop, the CLS query's softmax over the CLS key and
    the crop's patch keys, averaged over the heads.
    q_cls, k_cls: [B, C, H, dh]; k: [B, N, H, dh] (crop c = tokens c*N/C ..)."""
    q, kc, kp = _f32(q_cls), _f32(k_cls), _f32(k)
    B, C, H, dh = q.shape
    N = kp.shape[1]
    A = np.empty((B, N), np.float64)
    rc = _load().p4q_cls_saliency(_ptr(q), _ptr(kc), _ptr(kp), B, N, C, H, dh, _ptr(A))
    if rc != OK:
        raise ValueError(f"oracle cls_saliency failed ({rc})")
    return A


def swiglu_quantize_rows(gate, up):
    """h = silu(gate) * up (silu(g) = g / (1 + exp(-g)) in float64, rounded once to
    fp32), then the per-row 4-bit quantizer: returns (codes int8 [rows, cols],
    scale fp32 [rows])."""
    g, u = _f32(gate), _f32(up)
    assert g.shape == u.shape and g.ndim == 2
    rows, cols = g.shape
    codes = np.empty((rows, cols), np.int8)
    scale = np.empty((rows,), np.float32)
    rc = _load().p4q_swiglu_quantize_rows(_ptr(g), _ptr(u), rows, cols, _ptr(codes), _ptr(scale))
    if rc != OK:
        raise ValueError(f"oracle swiglu_quantize_rows failed ({rc})")
    return codes, scale


def sumsq32(x) -> np.float32:
    """The exact sum of squares of fp16 values, rounded once to fp32."""
    a = _f32(x).ravel()
    v = _load().oracle_sumsq32(_ptr(a), a.size)
    if v < 0:
        raise ValueError("oracle sumsq32: input is not fp16-valued")
    return np.float32(v)


def rmsnorm_rows(x, w, eps):
    """RMSNorm of each row of fp16 values x [rows, cols] with gain w [cols]
    (fp16 values): returns y as float32 [rows, cols] holding fp16 values."""
    a, g = _f32(x), _f32(w)
    assert a.ndim == 2 and g.shape == (a.shape[1],)
    y = np.empty_like(a)
    rc = _load().p4q_rmsnorm_rows(_ptr(a), _ptr(g), float(eps), a.shape[0], a.shape[1], _ptr(y))
    if rc != OK:
        raise ValueError(f"oracle rmsnorm_rows failed ({rc})")
    return y


def rmsnorm_quantize_rows(x, w, eps):
    """RMSNorm then the per-row 4-bit quantizer: (codes int8 [rows, cols], scale fp32 [rows])."""
    a, g = _f32(x), _f32(w)
    assert a.ndim == 2 and g.shape == (a.shape[1],)
    rows, cols = a.shape
    codes = np.empty((rows, cols), np.int8)
    scale = np.empty((rows,), np.float32)
    rc = _load().p4q_rmsnorm_quantize_rows(_ptr(a), _ptr(g), float(eps), rows, cols, _ptr(codes), _ptr(scale))
    if rc != OK:
        raise ValueError(f"oracle rmsnorm_quantize_rows failed ({rc})")
    return codes, scale


def causal_attention(q, k, v, B, m, H, Hkv, dh):
    """Causal softmax attention per sample and head (fp64): q [B*m, H*dh],
    k, v [B*m, Hkv*dh] (fp16 values); returns o float64 [B*m, H*dh]."""
    q, k, v = _f32(q), _f32(k), _f32(v)
    assert q.shape == (B * m, H * dh) and k.shape == (B * m, Hkv * dh) and v.shape == k.shape
    o = np.empty((B * m, H * dh), np.float64)
    rc = _load().p4q_causal_attention(_ptr(q), _ptr(k), _ptr(v), B, m, H, Hkv, dh, _ptr(o))
    if rc != OK:
        raise ValueError(f"oracle causal_attention failed ({rc})")
    return o


def block_mse(Yq, Yf, offsets):
    """Eq. 5's block objective: per-sample ||Yq - Yf||_F^2 / (m_n d) over rows
    offsets[n] .. offsets[n+1]-1, and their mean. Returns (e float64 [B], L)."""
    a, f = _f32(Yq), _f32(Yf)
    off = np.ascontiguousarray(offsets, np.int32)
    assert a.ndim == 2 and a.shape == f.shape and off[-1] == a.shape[0]
    B = off.size - 1
    e = np.empty(B, np.float64)
    L = np.empty(1, np.float64)
    rc = _load().p4q_block_mse(_ptr(a), _ptr(f), _ptr(off), B, a.shape[1], _ptr(e), _ptr(L))
    if rc != OK:
        raise ValueError(f"oracle block_mse failed ({rc})")
    return e, float(L[0])


def topk_replacement(s_ref, s_alt, K):
    """Eq. 9's replacement ratio per sample (Top-K sets, ties to the lower
    index): returns (intersection int32 [B], rho float32 [B])."""
    r, a = _f32(s_ref), _f32(s_alt)
    assert r.ndim == 2 and r.shape == a.shape
    B, N = r.shape
    inter = np.empty(B, np.int32)
    rho = np.empty(B, np.float32)
    rc = _load().p4q_topk_replacement(_ptr(r), _ptr(a), B, N, int(K), _ptr(inter), _ptr(rho))
    if rc != OK:
        raise ValueError(f"oracle topk_replacement failed ({rc})")
    return inter, rho


def pack_codes(codes):
    """Pack int8 codes in [-8, 7] two per byte: even index in the low nibble, two's complement.

    This is the storage layout of the packed INT4 tensors; the tests use it to
    compare the GPU's packed bytes with the oracle's codes.
    """
    c = np.asarray(codes, np.int8)
    assert c.shape[-1] % 2 == 0
    u = (c.astype(np.int16) & 0xF).astype(np.uint8)
    return (u[..., 0::2] | (u[..., 1::2] << 4)).astype(np.uint8)


def unpack_codes(packed):
    """Inverse of pack_codes: uint8 [..., n/2] -> int8 [..., n]."""
    p = np.asarray(packed, np.uint8)
    lo = (p & 0xF).astype(np.int16)
    hi = (p >> 4).astype(np.int16)
    lo = np.where(lo >= 8, lo - 16, lo)
    hi = np.where(hi >= 8, hi - 16, hi)
    out = np.empty(p.shape[:-1] + (p.shape[-1] * 2,), np.int8)
    out[..., 0::2] = lo
    out[..., 1::2] = hi
    return out
