"""Host-side checks of the C ABI (no GPU needed): the library builds, exports
every entry point include/p4q.h declares, and validates arguments before it
touches a device."""
import ctypes
import os
import re

import pytest

from paper_2609_34867_gb300 import build as B

HEADER = os.path.join(B.ROOT, "include", "p4q.h")


def declared_functions():
    text = open(HEADER).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(p4q_[a-z0-9_]+)\s*\(", text)))


@pytest.fixture(scope="module")
def lib():
    B.build()
    return ctypes.CDLL(B.LIB)


def test_header_declares_the_boundary():
    names = declared_functions()
    for required in ["p4q_select", "p4q_quant_act", "p4q_w4a4_linear", "p4q_select_gather_quant",
                     "p4q_quant_weight", "p4q_w4a4_gemm_s32", "p4q_select_workspace_bytes",
                     "p4q_status_string", "p4q_device_status"]:
        assert required in names


def test_library_exports_every_declared_symbol(lib):
    for name in declared_functions():
        assert hasattr(lib, name), name


def test_status_strings(lib):
    lib.p4q_status_string.restype = ctypes.c_char_p
    lib.p4q_status_string.argtypes = [ctypes.c_int]
    for s in range(8):
        assert lib.p4q_status_string(s)
    assert lib.p4q_status_string(0) == b"ok"


def test_invalid_arguments_are_rejected_before_any_launch(lib):
    P, I = ctypes.c_void_p, ctypes.c_int
    lib.p4q_quant_act.argtypes = [P, I, I, P, P, P]
    assert lib.p4q_quant_act(None, -1, 128, None, None, None) == 1         # negative M
    assert lib.p4q_quant_act(P(16), 4, 100, P(16), P(16), None) == 2      # Kin % 16
    assert lib.p4q_quant_act(P(8), 4, 128, P(16), P(16), None) == 3       # misaligned X
    assert lib.p4q_quant_act(None, 0, 128, None, None, None) == 0         # empty is a no-op
    lib.p4q_w4a4_linear.argtypes = [P, P, I, I, P, P, I, P, P]
    assert lib.p4q_w4a4_linear(P(16), P(16), 4, 100, P(16), P(16), 8, P(16), None) == 2   # Kin % 128
    assert lib.p4q_w4a4_linear(P(16), P(16), 4, 128, P(16), P(16), 12, P(16), None) == 2  # N % 8
    assert lib.p4q_w4a4_linear(P(16), P(16), 4, 128, None, P(16), 8, P(16), None) == 1


def test_cls_saliency_validates_shapes(lib):
    P, I = ctypes.c_void_p, ctypes.c_int
    lib.p4q_cls_saliency.argtypes = [P, P, P, I, I, I, I, I, P, P]
    f = lib.p4q_cls_saliency
    ok = (P(16), P(16), P(16))
    assert f(None, P(16), P(16), 1, 576, 1, 16, 64, P(16), None) == 1   # null pointer
    assert f(*ok, 0, 576, 1, 16, 64, P(16), None) == 1                  # B < 1
    assert f(*ok, 1, 577, 2, 16, 64, P(16), None) == 2                  # N % C
    assert f(*ok, 1, 576, 1, 16, 48, P(16), None) == 2                  # head dim
    assert f(*ok, 1, 576, 1, 33, 64, P(16), None) == 2                  # heads
    assert f(*ok, 1, 4096, 1, 32, 64, P(16), None) == 2                 # one crop's weights exceed shared memory
    assert f(P(8), P(16), P(16), 1, 576, 1, 16, 64, P(16), None) == 3   # misaligned


def test_swiglu_quant_validates_arguments(lib):
    P, I = ctypes.c_void_p, ctypes.c_int
    lib.p4q_swiglu_quant_expanded.argtypes = [P, I, P, I, I, I, P, P, P, P, P]
    f = lib.p4q_swiglu_quant_expanded
    assert f(P(16), 4096, P(16), 4096, 0, 4096, P(16), P(16), None, None, None) == 0     # empty is a no-op
    assert f(P(16), 4096, P(16), 4096, 4, 4096, P(16), P(16), P(16), None, None) == 1    # Xu without sum_xu
    assert f(P(16), 100, P(16), 4096, 4, 4096, P(16), P(16), None, None, None) == 1      # pitch < Kin
    assert f(P(16), 4096, P(16), 4096, 4, 4100, P(16), P(16), None, None, None) == 1     # pitch < Kin
    assert f(P(16), 4104, P(16), 4104, 4, 4100, P(16), P(16), None, None, None) == 2     # Kin % 16
    assert f(P(16), 4100, P(16), 4104, 4, 4096, P(16), P(16), None, None, None) == 3     # pitch % 8
    assert f(P(8), 4096, P(16), 4096, 4, 4096, P(16), P(16), None, None, None) == 3      # misaligned gate


def test_rmsnorm_quant_validates_arguments(lib):
    P, I, F = ctypes.c_void_p, ctypes.c_int, ctypes.c_float
    lib.p4q_rmsnorm_quant_expanded.argtypes = [P, I, P, F, I, I, P, P, P, P, P]
    f = lib.p4q_rmsnorm_quant_expanded
    assert f(P(16), 4096, P(16), 1e-6, 0, 4096, P(16), P(16), None, None, None) == 0     # empty is a no-op
    assert f(P(16), 4096, P(16), 1e-6, 4, 4096, P(16), P(16), P(16), None, None) == 1    # Xu without sum_xu
    assert f(P(16), 4096, P(16), -1.0, 4, 4096, P(16), P(16), None, None, None) == 1     # eps < 0
    assert f(P(16), 4096, P(16), float("nan"), 4, 4096, P(16), P(16), None, None, None) == 1
    assert f(P(16), 4096, P(16), float("inf"), 4, 4096, P(16), P(16), None, None, None) == 1
    assert f(P(16), 4096, None, 1e-6, 4, 4096, P(16), P(16), None, None, None) == 1      # no gain
    assert f(P(16), 100, P(16), 1e-6, 4, 4096, P(16), P(16), None, None, None) == 1      # pitch < Kin
    assert f(P(16), 4104, P(16), 1e-6, 4, 4100, P(16), P(16), None, None, None) == 2     # Kin % 16
    assert f(P(16), 4100, P(16), 1e-6, 4, 4096, P(16), P(16), None, None, None) == 3     # pitch % 8
    assert f(P(16), 4096, P(8), 1e-6, 4, 4096, P(16), P(16), None, None, None) == 3      # misaligned gain


def test_causal_attention_validates_arguments(lib):
    P, I = ctypes.c_void_p, ctypes.c_int
    lib.p4q_causal_attention.argtypes = [P, I, P, I, P, I, I, I, I, I, I, P, I, P]
    f = lib.p4q_causal_attention
    ok = (P(16), 4096, P(16), 4096, P(16), 4096)
    assert f(*ok, 0, 256, 32, 32, 128, P(16), 4096, None) == 0        # empty is a no-op
    assert f(*ok, 2, 0, 32, 32, 128, P(16), 4096, None) == 1          # m < 1
    assert f(*ok, 2, 256, 32, 5, 128, P(16), 4096, None) == 1         # H % Hkv
    assert f(*ok, 2, 256, 32, 32, 128, P(16), 2048, None) == 1        # ldo < H dh
    assert f(*ok, 2, 256, 32, 32, 128, None, 4096, None) == 1         # no output
    assert f(*ok, 2, 256, 32, 32, 64, P(16), 4096, None) == 2         # dh != 128
    assert f(*ok, 2, 8193, 32, 32, 128, P(16), 4096, None) == 2       # m > 8192
    assert f(P(16), 4100, P(16), 4096, P(16), 4096, 2, 256, 32, 32, 128, P(16), 4096, None) == 3  # pitch % 8
    assert f(P(8), 4096, P(16), 4096, P(16), 4096, 2, 256, 32, 32, 128, P(16), 4096, None) == 3   # misaligned


def test_calibration_entries_validate_arguments(lib):
    P, I, S = ctypes.c_void_p, ctypes.c_int, ctypes.c_size_t
    lib.p4q_block_mse_workspace_bytes.argtypes = [I]
    lib.p4q_block_mse_workspace_bytes.restype = S
    assert lib.p4q_block_mse_workspace_bytes(0) == 0 and lib.p4q_block_mse_workspace_bytes(1025) == 0
    assert lib.p4q_block_mse_workspace_bytes(8) >= 8 * 8
    lib.p4q_block_mse.argtypes = [P, I, P, I, P, I, I, P, P, P, S, P]
    f = lib.p4q_block_mse
    off = (ctypes.c_int32 * 3)(0, 10, 20)
    bad = (ctypes.c_int32 * 3)(0, 10, 10)
    first = (ctypes.c_int32 * 3)(1, 10, 20)
    big = 1 << 20
    assert f(P(16), 64, P(16), 64, bad, 2, 64, P(16), P(16), P(16), big, None) == 1    # empty sample
    assert f(P(16), 64, P(16), 64, first, 2, 64, P(16), P(16), P(16), big, None) == 1  # offsets[0] != 0
    assert f(P(16), 64, P(16), 64, None, 2, 64, P(16), P(16), P(16), big, None) == 1   # no offsets
    assert f(P(16), 64, P(16), 64, off, 2, 60, P(16), P(16), P(16), big, None) == 2    # d % 8
    assert f(P(16), 68, P(16), 64, off, 2, 64, P(16), P(16), P(16), big, None) == 3    # pitch % 8
    assert f(P(16), 64, P(16), 64, off, 2, 64, P(16), P(16), P(16), 8, None) == 4      # workspace
    lib.p4q_topk_replacement.argtypes = [P, P, I, I, I, P, P, P]
    g = lib.p4q_topk_replacement
    assert g(P(16), P(16), 0, 576, 64, P(16), P(16), None) == 0       # empty is a no-op
    assert g(P(16), P(16), 2, 576, 577, P(16), P(16), None) == 1      # K > N
    assert g(P(16), P(16), 2, 576, 0, P(16), P(16), None) == 1        # K < 1
    assert g(None, P(16), 2, 576, 64, P(16), P(16), None) == 1        # no scores
    assert g(P(16), P(16), 2, 4097, 64, P(16), P(16), None) == 2      # N > P4Q_MAX_TOKENS


class Params(ctypes.Structure):
    _fields_ = [("K", ctypes.c_int32), ("alpha_permille", ctypes.c_int32), ("beta_permille", ctypes.c_int32)]


def test_workspace_query_and_select_validation(lib):
    P, I = ctypes.c_void_p, ctypes.c_int
    lib.p4q_select_workspace_bytes.argtypes = [I, I, I, I, ctypes.POINTER(Params)]
    lib.p4q_select_workspace_bytes.restype = ctypes.c_size_t
    p = Params(64, 300, 200)
    n = lib.p4q_select_workspace_bytes(1, 576, 4096, 3, ctypes.byref(p))
    assert n > 576 * 576 * 4 and n % 256 == 0
    assert lib.p4q_select_workspace_bytes(1, 576, 4000, 3, ctypes.byref(p)) == 0   # d % 128
    bad = Params(700, 300, 200)
    assert lib.p4q_select_workspace_bytes(1, 576, 4096, 3, ctypes.byref(bad)) == 0  # K > N
    lib.p4q_select.argtypes = [P, I, I, I, P, I, P, ctypes.POINTER(Params), P, P, ctypes.c_size_t, P]
    assert lib.p4q_select(P(16), 1, 576, 4096, None, 0, None, ctypes.byref(bad), P(16), P(256), 0, None) == 1
    over = Params(64, 800, 300)
    assert lib.p4q_select(P(16), 1, 576, 4096, None, 0, None, ctypes.byref(over), P(16), P(256), 0, None) == 1


def test_no_device_is_reported_not_faked(lib):
    """Without an sm_103 device a valid call returns P4Q_ERR_NO_DEVICE instead of computing on the CPU."""
    import torch
    if torch.cuda.is_available():
        pytest.skip("a GPU is present")
    P, I = ctypes.c_void_p, ctypes.c_int
    lib.p4q_quant_act.argtypes = [P, I, I, P, P, P]
    assert lib.p4q_quant_act(P(16), 4, 128, P(16), P(16), None) == 7


def test_wait_timeout_test_entry_validates_its_limit(lib):
    lib.p4q_test_wait_timeout.argtypes = [ctypes.c_uint32, ctypes.c_void_p]
    assert lib.p4q_test_wait_timeout(0, None) == 1
    assert lib.p4q_test_wait_timeout(1000001, None) == 1


def test_peak_probe_validates_its_arguments(lib):
    P, I = ctypes.c_void_p, ctypes.c_int
    lib.p4q_peak_probe.argtypes = [I, I, P, ctypes.POINTER(ctypes.c_double), P]
    ops = ctypes.c_double(0.0)
    assert lib.p4q_peak_probe(3, 10, P(16), ctypes.byref(ops), None) == 1        # unknown kind
    assert lib.p4q_peak_probe(0, 0, P(16), ctypes.byref(ops), None) == 1         # no iterations
    assert lib.p4q_peak_probe(1, 1 << 25, P(16), ctypes.byref(ops), None) == 1   # beyond the limit
    assert lib.p4q_peak_probe(2, 10, None, ctypes.byref(ops), None) == 1         # no sink
    assert lib.p4q_peak_probe(2, 10, P(16), None, None) == 1                     # no ops pointer
    assert lib.p4q_peak_probe(2, 10, P(20), ctypes.byref(ops), None) == 3        # sink misaligned


def test_strided_quantizer_validates_its_row_pitch(lib):
    P, I = ctypes.c_void_p, ctypes.c_int
    lib.p4q_quant_act_ld.argtypes = [P, I, I, I, P, P, P]
    assert lib.p4q_quant_act_ld(P(16), 64, 4, 128, P(16), P(16), None) == 1   # pitch below the row length
    assert lib.p4q_quant_act_ld(P(16), 132, 4, 128, P(16), P(16), None) == 3  # rows not 16-byte aligned
    assert lib.p4q_quant_act_ld(None, 128, 0, 128, None, None, None) == 0     # empty is a no-op


def test_rowmax_entries_validate_their_blocks(lib):
    P, I = ctypes.c_void_p, ctypes.c_int
    ints = lambda *v: (ctypes.c_int * len(v))(*v)
    ptrs = lambda *v: (ctypes.c_void_p * len(v))(*v)
    g = lib.p4q_w4a4_linear_expanded_rowmax
    g.argtypes = [P, P, P, I, I, P, P, P, I, P, I, P, P, P, P]
    a = (P(16), P(16), P(16), 4, 128, P(16), P(16), P(16), 512, P(16))
    assert g(*a, 3, ints(0, 0, 0), ints(32, 32, 32), P(16), None) == 1          # at most two blocks
    assert g(*a, 1, ints(480), ints(64), P(16), None) == 1                      # past N
    assert g(*a, 1, ints(16), ints(64), P(16), None) == 2                       # not a multiple of 32
    assert g(*a, 1, ints(0), ints(64), None, None) == 1                         # no rowmax
    assert g(P(16), P(16), P(16), 0, 128, P(16), P(16), P(16), 512, P(16), 1, ints(0), ints(64), None,
             None) == 0                                                          # M == 0 is a no-op
    q = lib.p4q_quant_act_expanded_rowmax
    q.argtypes = [P, I, I, I, P, P, P, P, P, P, P, P]
    sinks = (ptrs(16, 16), ptrs(16, 16), ptrs(16, 16), ptrs(16, 16))
    assert q(P(16), 1024, 4, 2, ints(0, 512), ints(256, 384), P(16), *sinks, None) == 2   # 384 % 256
    assert q(P(16), 1024, 4, 2, ints(0, 896), ints(256, 256), P(16), *sinks, None) == 1   # past ldy
    assert q(P(16), 1024, 4, 1, ints(4), ints(256), P(16), *sinks, None) == 3             # col0 % 8
    assert q(P(16), 1024, 4, 1, ints(0), ints(256), P(16), ptrs(16), ptrs(8), ptrs(16), ptrs(16),
             None) == 3                                                                  # misaligned s_a
    assert q(P(16), 1024, 0, 1, ints(0), ints(256), None, None, ptrs(16), ptrs(16), ptrs(16),
             None) == 0                                                                  # M == 0
