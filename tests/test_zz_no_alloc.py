"""p4q_select_noalloc: the selector for callers that cannot allocate device
memory when they select (for example a runtime that owns the allocator and
hands the library only its inputs and outputs). Its scratch is a fixed array
inside the library, so it must give the indices of the oracle and of
p4q_select with a caller workspace, call after call, up to the largest batch
the array holds, and refuse the next size up before launching anything.

Collected last (file name) so that a failure here comes after every other test.
"""
import ctypes

import numpy as np
import pytest
import torch

import oracle
from paper_2609_34867_gb300 import workloads as wl

pytestmark = pytest.mark.gpu

SCRATCH = 48 << 20  # P4Q_NOALLOC_SCRATCH_BYTES
TOO_SMALL = 4       # P4Q_ERR_WORKSPACE_TOO_SMALL


class Params(ctypes.Structure):
    _fields_ = [("K", ctypes.c_int32), ("alpha_permille", ctypes.c_int32), ("beta_permille", ctypes.c_int32)]


def _fn(lib):
    P, I = ctypes.c_void_p, ctypes.c_int
    f = lib.p4q_select_noalloc
    f.argtypes = [P, I, I, I, P, I, P, ctypes.POINTER(Params), P, P]
    f.restype = ctypes.c_int
    return f


def _call(f, V, Q, A, K, idx, stream):
    B, N, d = V.shape
    p = Params(K, 300, 200)
    return f(ctypes.c_void_p(V.data_ptr()), B, N, d, ctypes.c_void_p(Q.data_ptr()), Q.shape[1],
             ctypes.c_void_p(A.data_ptr()), ctypes.byref(p), ctypes.c_void_p(idx.data_ptr()),
             ctypes.c_void_p(stream.cuda_stream))


def test_noalloc_select_matches_workspace_select_twice(p4q, dev):
    f = _fn(p4q.lib())
    stream = torch.cuda.current_stream()
    for seed, (B, N, d, K) in enumerate([(2, 300, 256, 40), (3, 576, 512, 64)]):
        w = wl.Workload("t", B=B, N=N, d=d, K=K, T=0, J=3, seed=seed + 30, heavy_tail=False, linears=())
        x = wl.selector_inputs(w)
        V, Q, A = (torch.from_numpy(a).to(dev) for a in (x.V, x.Q, x.A))
        ref = p4q.select(V, Q, A, K).cpu().numpy()  # the existing entry point, caller workspace
        for _ in range(2):  # two calls in a row share the same scratch
            idx = torch.full((B, K), -1, dtype=torch.int32, device=dev)
            assert _call(f, V, Q, A, K, idx, stream) == 0
            torch.cuda.synchronize()
            assert p4q.p4q_device_status() == 0
            assert np.array_equal(idx.cpu().numpy(), ref)


def test_noalloc_select_at_its_capacity_and_just_beyond(p4q, dev):
    """LLaVA-1.5 images (576 x 4096, 3 concepts, K = 192): the largest batch the
    scratch holds runs, twice, and equals the oracle and the workspace call; one
    image more is refused with P4Q_ERR_WORKSPACE_TOO_SMALL."""
    f = _fn(p4q.lib())
    stream = torch.cuda.current_stream()
    N, d, K = 576, 4096, 192
    w = wl.Workload("t", B=40, N=N, d=d, K=K, T=0, J=3, seed=44, heavy_tail=False, linears=())
    x = wl.selector_inputs(w)
    Vall, Qall, Aall = (torch.from_numpy(a).to(dev) for a in (x.V, x.Q, x.A))
    fits, refused = None, None
    for B in range(1, 41):  # rejected sizes launch nothing, so probing them is safe
        idx = torch.full((B, K), -1, dtype=torch.int32, device=dev)
        rc = _call(f, Vall[:B], Qall[:B], Aall[:B], K, idx, stream)
        torch.cuda.synchronize()
        if rc == TOO_SMALL:
            refused = B
            break
        assert rc == 0
        fits = (B, idx)
    assert fits is not None and refused == fits[0] + 1, (fits and fits[0], refused)
    B = fits[0]
    assert B >= 8, "the documented capacity (8 LLaVA-1.5 images) does not fit"
    # the size query is an upper bound of what a call needs
    assert p4q.p4q_select_workspace_bytes(B + 1, N, d, 3, K) > SCRATCH
    assert p4q.p4q_device_status() == 0
    ref = oracle.select_batch(x.V[:B], K, x.Q[:B], x.A[:B])
    assert np.array_equal(fits[1].cpu().numpy(), ref)
    assert np.array_equal(p4q.select(Vall[:B], Qall[:B], Aall[:B], K).cpu().numpy(), ref)
    idx = torch.full((B, K), -1, dtype=torch.int32, device=dev)
    assert _call(f, Vall[:B], Qall[:B], Aall[:B], K, idx, stream) == 0  # a second call on the same scratch
    torch.cuda.synchronize()
    assert np.array_equal(idx.cpu().numpy(), ref)


def test_noalloc_select_rejects_sizes_beyond_its_scratch(p4q, dev):
    f = _fn(p4q.lib())
    B, N, d, K = 64, 2880, 4096, 320  # workspace of several GB, far above the fixed scratch
    need = p4q.p4q_select_workspace_bytes(B, N, d, 3, K)
    assert need > SCRATCH
    V = torch.zeros((1, 1, 16), dtype=torch.float16, device=dev)  # never read: rejected before any launch
    Q = torch.zeros((1, 1, 16), dtype=torch.float16, device=dev)
    A = torch.zeros((1, 1), dtype=torch.float32, device=dev)
    idx = torch.zeros((1, 1), dtype=torch.int32, device=dev)
    p = Params(K, 300, 200)
    rc = f(ctypes.c_void_p(V.data_ptr()), B, N, d, ctypes.c_void_p(Q.data_ptr()), 3, ctypes.c_void_p(A.data_ptr()),
           ctypes.byref(p), ctypes.c_void_p(idx.data_ptr()), ctypes.c_void_p(torch.cuda.current_stream().cuda_stream))
    assert rc == TOO_SMALL
