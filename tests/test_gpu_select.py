"""GPU parity of the quantization-aware selector (Sec. 3.2, Eq. 4) and of the
fused gather + quantize against the oracle: kept index sets identical,
gathered rows and their INT4 codes / scales bit-exact."""
import numpy as np
import pytest
import torch

import oracle
from paper_2609_34867_gb300 import workloads as wl

pytestmark = pytest.mark.gpu


def _t(x, dev):
    return None if x is None else torch.from_numpy(np.ascontiguousarray(x)).to(dev)


def _select(p4q, dev, x, K, use_q=True, use_a=True, alpha=300, beta=200):
    Q = x.Q if use_q else None
    A = x.A if use_a else None
    idx = p4q.select(_t(x.V, dev), _t(Q, dev), _t(A, dev), K, alpha_permille=alpha, beta_permille=beta)
    torch.cuda.synchronize()
    assert p4q.p4q_device_status() == 0
    ref = oracle.select_batch(x.V, K, Q, A, alpha, beta)
    return idx.cpu().numpy(), ref


@pytest.mark.parametrize("B,N,d,K,J,seed", [(2, 100, 128, 20, 3, 0), (3, 576, 256, 64, 3, 1),
                                            (1, 30, 128, 10, 2, 2), (2, 301, 384, 77, 5, 3),
                                            (1, 1152, 128, 200, 3, 4),
                                            (1, 2048, 5376, 160, 2, 5)])  # rows wider than the token pass
def test_select_matches_oracle(p4q, dev, B, N, d, K, J, seed):
    w = wl.Workload("t", B=B, N=N, d=d, K=K, T=0, J=J, seed=seed, heavy_tail=False, linears=())
    got, ref = _select(p4q, dev, wl.selector_inputs(w), K)
    assert np.array_equal(got, ref)


@pytest.mark.parametrize("use_q,use_a,alpha,beta", [(False, True, 300, 200), (True, False, 300, 200),
                                                    (False, False, 300, 200), (True, True, 0, 0),
                                                    (True, True, 1000, 0), (True, True, 0, 1000)])
def test_select_signal_variants(p4q, dev, use_q, use_a, alpha, beta):
    w = wl.Workload("t", B=2, N=200, d=256, K=40, T=0, J=3, seed=9, heavy_tail=True, linears=())
    got, ref = _select(p4q, dev, wl.selector_inputs(w), 40, use_q, use_a, alpha, beta)
    assert np.array_equal(got, ref)


@pytest.mark.parametrize("K", [1, 576])
def test_select_budget_extremes(p4q, dev, K):
    w = wl.Workload("t", B=1, N=576, d=128, K=K, T=0, J=3, seed=5, heavy_tail=False, linears=())
    got, ref = _select(p4q, dev, wl.selector_inputs(w), K)
    assert np.array_equal(got, ref)


def test_select_orthogonal_ties(p4q, dev):
    """All cosines 0: every diversity pick is a tie won by the lowest index."""
    N, d = 130, 256
    V = np.zeros((1, N, d), np.float16)
    V[0, np.arange(N), np.arange(N)] = 1.0
    idx = p4q.select(_t(V, dev), None, None, 17)
    assert np.array_equal(idx.cpu().numpy()[0], np.arange(17))


def _clustered(B, N, d, centers, seed, noise=0.05):
    """Tokens drawn around a few centres: a pick raises the diversity maxima
    of its whole cluster, so the greedy rounds run in many short phases."""
    rng = np.random.default_rng(seed)
    C = rng.standard_normal((B, centers, d)).astype(np.float32)
    lab = rng.integers(0, centers, size=(B, N))
    V = np.take_along_axis(C, lab[:, :, None], axis=1) + noise * rng.standard_normal((B, N, d)).astype(np.float32)
    return V.astype(np.float16)


@pytest.mark.parametrize("use_signals", [False, True])
def test_select_clustered_tokens_many_phases(p4q, dev, use_signals):
    B, N, d, K = 2, 600, 256, 300
    V = _clustered(B, N, d, 40, seed=21)
    rng = np.random.default_rng(22)
    Q = V[:, rng.integers(0, N, 3)].astype(np.float16) if use_signals else None
    A = rng.random((B, N)).astype(np.float32) if use_signals else None
    idx = p4q.select(_t(V, dev), _t(Q, dev), _t(A, dev), K)
    torch.cuda.synchronize()
    assert p4q.p4q_device_status() == 0
    ref = oracle.select_batch(V, K, Q, A)
    assert np.array_equal(idx.cpu().numpy(), ref)


def test_select_duplicate_tokens(p4q, dev):
    """Every token appears three times: a pick's copies reach cosine 1 and are
    kept only after every other token; ties resolve to the lower index."""
    rng = np.random.default_rng(23)
    base = rng.standard_normal((1, 100, 128)).astype(np.float32)
    V = np.concatenate([base, base, base], axis=1).astype(np.float16)
    for K in (90, 150, 250):
        idx = p4q.select(_t(V, dev), None, None, K)
        torch.cuda.synchronize()
        assert p4q.p4q_device_status() == 0
        assert np.array_equal(idx.cpu().numpy(), oracle.select_batch(V, K))


@pytest.mark.parametrize("N,K,d", [(2880, 640, 256), (4096, 1024, 128), (2049, 2000, 128), (4096, 2048, 128),
                                   (4096, 2400, 128)])
def test_select_large_token_sets(p4q, dev, N, K, d):
    """Block sizes of 768 and 1024 ranking threads, several column chunks per
    pool phase (up to K_d picks unseen by a pool), K close to N; kept sets R0
    of 320, 512, 1000 and 1024 tokens (two to four column tiles of the
    cosine-max epilogue) and 1200 (int32 tiles and the row pass)."""
    w = wl.Workload("t", B=2, N=N, d=d, K=K, T=0, J=3, seed=31, heavy_tail=True, linears=())
    got, ref = _select(p4q, dev, wl.selector_inputs(w), K)
    assert np.array_equal(got, ref)


def test_select_one_image_576_tokens_4096d(p4q, dev):
    """The single-image LLaVA-1.5 shape: 576 tokens x 4096, budget 64."""
    w = wl.LLAVA15_7B_ONE
    got, ref = _select(p4q, dev, wl.selector_inputs(w), w.K)
    assert np.array_equal(got, ref)


def test_select_gather_quant_matches_oracle(p4q, dev):
    w = wl.Workload("t", B=3, N=320, d=512, K=48, T=16, J=3, seed=7, heavy_tail=False, linears=())
    x = wl.selector_inputs(w)
    idx, X, Xq, s_a = p4q.select_gather_quant(_t(x.V, dev), _t(x.Q, dev), _t(x.A, dev), _t(x.text, dev), w.K)
    torch.cuda.synchronize()
    ref_idx = oracle.select_batch(x.V, w.K, x.Q, x.A)
    assert np.array_equal(idx.cpu().numpy(), ref_idx)
    Xr = oracle.gather(x.V, ref_idx, x.text)
    assert np.array_equal(X.cpu().numpy().astype(np.float32), Xr)
    c, s = oracle.quantize_rows(Xr.reshape(-1, w.d))
    assert np.array_equal(oracle.unpack_codes(Xq.cpu().numpy()), c)
    assert np.array_equal(s_a.cpu().numpy().view(np.uint32), s.view(np.uint32))


def test_select_gather_quant_without_text(p4q, dev):
    w = wl.Workload("t", B=2, N=200, d=256, K=30, T=0, J=3, seed=8, heavy_tail=False, linears=())
    x = wl.selector_inputs(w)
    idx, X, Xq, s_a = p4q.select_gather_quant(_t(x.V, dev), _t(x.Q, dev), _t(x.A, dev), None, w.K)
    torch.cuda.synchronize()
    ref_idx = oracle.select_batch(x.V, w.K, x.Q, x.A)
    assert np.array_equal(idx.cpu().numpy(), ref_idx)
    assert np.array_equal(X.cpu().numpy().astype(np.float32), oracle.gather(x.V, ref_idx))


def test_select_gather_quant_expanded_matches(p4q, dev):
    w = wl.Workload("t", B=2, N=300, d=512, K=40, T=8, J=3, seed=17, heavy_tail=False, linears=())
    x = wl.selector_inputs(w)
    V, Q, A, T = (_t(a, dev) for a in (x.V, x.Q, x.A, x.text))
    ws = p4q.select_workspace(w.B, w.N, w.d, w.J, w.K, dev)
    M = w.B * (w.K + w.T)
    idx = torch.empty((w.B, w.K), dtype=torch.int32, device=dev)
    X = torch.empty((w.B, w.K + w.T, w.d), dtype=torch.float16, device=dev)
    Xq = torch.empty((M, w.d // 2), dtype=torch.uint8, device=dev)
    s = torch.empty((M,), dtype=torch.float32, device=dev)
    Xu = torch.empty((M, w.d), dtype=torch.uint8, device=dev)
    su = torch.empty((M,), dtype=torch.int32, device=dev)
    p4q.p4q_select_gather_quant_expanded(V, Q, A, T, w.K, idx, X, Xq, s, Xu, su, ws)
    ref_idx, ref_X, ref_q, ref_s = p4q.select_gather_quant(V, Q, A, T, w.K)
    ref_u, ref_su = p4q.expand_codes(ref_q)
    torch.cuda.synchronize()
    assert torch.equal(idx, ref_idx) and torch.equal(X.view(torch.int16), ref_X.view(torch.int16))
    assert torch.equal(Xq, ref_q) and torch.equal(Xu, ref_u) and torch.equal(su, ref_su)


def test_select_gather_quant_expanded_nine_images_matches_oracle(p4q, dev):
    """Nine images of more than 1024 tokens (no Gram mode: the kept set's
    cosine-max GEMM and the candidates' pair GEMM), twice on the same
    workspace: every image's indices, gathered rows, codes, scales and
    expanded codes against the oracle."""
    w = wl.Workload("t", B=9, N=1100, d=256, K=150, T=12, J=3, seed=23, heavy_tail=False, linears=())
    x = wl.selector_inputs(w)
    V, Q, A, T = (_t(a, dev) for a in (x.V, x.Q, x.A, x.text))
    ws = p4q.select_workspace(w.B, w.N, w.d, w.J, w.K, dev)
    M = w.B * (w.K + w.T)
    idx = torch.full((w.B, w.K), -1, dtype=torch.int32, device=dev)
    X = torch.empty((w.B, w.K + w.T, w.d), dtype=torch.float16, device=dev)
    Xq = torch.empty((M, w.d // 2), dtype=torch.uint8, device=dev)
    s = torch.empty((M,), dtype=torch.float32, device=dev)
    Xu = torch.empty((M, w.d), dtype=torch.uint8, device=dev)
    su = torch.empty((M,), dtype=torch.int32, device=dev)
    for _ in range(2):
        p4q.p4q_select_gather_quant_expanded(V, Q, A, T, w.K, idx, X, Xq, s, Xu, su, ws)
    ref_u, ref_su = p4q.expand_codes(Xq)
    torch.cuda.synchronize()
    assert p4q.p4q_device_status() == 0
    ref_idx = oracle.select_batch(x.V, w.K, x.Q, x.A)
    assert np.array_equal(idx.cpu().numpy(), ref_idx)
    Xr = oracle.gather(x.V, ref_idx, x.text)
    assert np.array_equal(X.cpu().numpy().astype(np.float32), Xr)
    c, sr = oracle.quantize_rows(Xr.reshape(-1, w.d))
    assert np.array_equal(oracle.unpack_codes(Xq.cpu().numpy()), c)
    assert np.array_equal(s.cpu().numpy().view(np.uint32), sr.view(np.uint32))
    assert torch.equal(Xu, ref_u) and torch.equal(su, ref_su)


def test_select_from_two_host_threads_on_two_streams(p4q, dev):
    """Concurrent calls from two host threads on two streams, each with its own
    workspace: the library keeps no state between the launches of a call, so
    each call must see only its own inputs, call after call."""
    import threading

    cases = []
    for seed in (40, 41):
        w = wl.Workload("t", B=4, N=576, d=512, K=96, T=0, J=3, seed=seed, heavy_tail=False, linears=())
        x = wl.selector_inputs(w)
        ref = oracle.select_batch(x.V, w.K, x.Q, x.A)
        ins = (_t(x.V, dev), _t(x.Q, dev), _t(x.A, dev))
        cases.append((ins, w.K, ref))
    errors = []

    def run(i):
        try:
            (V, Q, A), K, ref = cases[i]
            stream = torch.cuda.Stream(device=dev)
            ws = p4q.select_workspace(V.shape[0], V.shape[1], V.shape[2], Q.shape[1], K, dev)
            for _ in range(20):
                with torch.cuda.stream(stream):
                    idx = torch.full((V.shape[0], K), -1, dtype=torch.int32, device=dev)
                    p4q.p4q_select(V, Q, A, K, idx, ws, stream=stream)
                stream.synchronize()
                if not np.array_equal(idx.cpu().numpy(), ref):
                    errors.append(i)
                    return
        except Exception as e:  # surfaced below
            errors.append(repr(e))

    torch.cuda.synchronize()  # the inputs are in place before either thread starts
    threads = [threading.Thread(target=run, args=(i,)) for i in range(2)]
    for t in threads:
        t.start()
    for t in threads:
        t.join()
    assert p4q.p4q_device_status() == 0
    assert not errors, errors
