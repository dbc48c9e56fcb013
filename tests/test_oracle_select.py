"""Pins for the oracle's three-stage selector (Sec. 3.2, Eq. 4), CPU only.

The selector is a greedy procedure, not an optimum of an objective, so it is
pinned by properties each stage must have, checked with float64 numpy cosines
of the dequantized fake-quantized vectors (computed here, not by the oracle),
by closed-form special cases, and by the budget split fixed by the paper's
alpha / beta / gamma and token budgets.
"""
import os

import numpy as np
import pytest

import oracle
from paper_2609_34867_gb300 import workloads as wl

TOL = 2e-6  # float64 cosine vs the oracle's fp32 cosine


def _deq(x):
    c, s = oracle.quantize_rows(x)
    return c.astype(np.float64) * s[:, None].astype(np.float64)


def _cos64(a, b):
    na = np.linalg.norm(a, axis=-1)
    nb = np.linalg.norm(b, axis=-1)
    den = np.outer(na, nb)
    g = a @ b.T
    return np.where(den > 0, g / np.where(den > 0, den, 1), 0.0)


def test_budget_split_golden(golden_dir):
    n = 0
    for line in open(os.path.join(golden_dir, "budget_split.txt")):
        line = line.strip()
        if not line or line.startswith("#"):
            continue
        K, kq, ks, kd = (int(v) for v in line.split())
        assert oracle.budget(K) == (kq, ks, kd)
        n += 1
    assert n >= 4
    # budget reassignment when a signal is absent
    assert oracle.budget(64, have_q=False) == (0, 12, 52)
    assert oracle.budget(64, have_a=False) == (19, 0, 45)
    assert oracle.budget(64, have_q=False, have_a=False) == (0, 0, 64)


def test_paper_pruning_ratios():
    """576 -> 64 and 2880 -> 320 both prune 88.9% of the visual tokens (Sec. 4, Table 1)."""
    assert round(100 * (1 - wl.LLAVA15_7B_ONE.K / wl.LLAVA15_7B_ONE.N), 1) == 88.9
    assert round(100 * (1 - wl.LLAVANEXT_7B.K / wl.LLAVANEXT_7B.N), 1) == 88.9


def _check_stages(V, Q, A, K, alpha=300, beta=200):
    idx, order, stage = oracle.select_one(V, K, Q, A, alpha, beta)
    N = V.shape[0]
    # invariants
    assert idx.shape == (K,) and len(set(idx.tolist())) == K
    assert np.all(np.diff(idx) > 0) and idx.min() >= 0 and idx.max() < N
    assert np.array_equal(np.sort(order), idx)
    kq, ks, kd = oracle.budget(K, alpha, beta, Q is not None, A is not None)
    assert (stage > 0).sum() == kq and (stage == -1).sum() == ks and (stage == -2).sum() == kd
    dv = _deq(V)
    kept = np.zeros(N, bool)
    t = 0
    # stage 1: per concept, its picks are the best remaining cosines
    if Q is not None:
        dq = _deq(Q)
        J = Q.shape[0]
        for j in range(J):
            quota = kq // J + (1 if j < kq % J else 0)
            score = _cos64(dq[j:j + 1], dv)[0]
            for _ in range(quota):
                p = order[t]
                assert stage[t] == 1 + j and not kept[p]
                assert score[p] >= score[~kept].max() - TOL
                kept[p] = True
                t += 1
    # stage 2: saliency on the rest, exact fp32 comparisons, lower index on ties
    for _ in range(ks):
        p = order[t]
        assert stage[t] == -1 and not kept[p]
        rest = np.where(~kept)[0]
        best = rest[np.argmax(A[rest])]  # argmax returns the first (lowest) index on ties
        assert p == best
        kept[p] = True
        t += 1
    # stage 3: each pick has the smallest max-cosine to the kept set
    G = _cos64(dv, dv)
    for _ in range(kd):
        p = order[t]
        assert stage[t] == -2 and not kept[p]
        rest = np.where(~kept)[0]
        if kept.any():
            m = G[np.ix_(rest, np.where(kept)[0])].max(axis=1)
            mp = G[p, kept].max()
            assert mp <= m.min() + TOL
        else:
            assert p == rest[0]
        kept[p] = True
        t += 1
    return idx, order, stage


@pytest.mark.parametrize("seed,N,d,K,J", [(0, 48, 64, 16, 3), (1, 96, 128, 40, 2),
                                          (2, 30, 32, 30, 3), (3, 64, 96, 7, 5)])
def test_stage_properties_random(seed, N, d, K, J):
    w = wl.Workload("t", B=1, N=N, d=d, K=K, T=0, J=J, seed=seed, heavy_tail=False, linears=())
    x = wl.selector_inputs(w)
    _check_stages(x.V[0], x.Q[0], x.A[0], K)


def test_stage_properties_without_signals():
    w = wl.Workload("t", B=1, N=80, d=64, K=24, T=0, J=3, seed=9, heavy_tail=True, linears=())
    x = wl.selector_inputs(w)
    _check_stages(x.V[0], None, x.A[0], 24)
    _check_stages(x.V[0], x.Q[0], None, 24)
    _check_stages(x.V[0], None, None, 24)


def test_orthogonal_one_hot_tokens_give_ascending_prefix():
    """All cosines are 0, so every diversity round is a tie won by the lowest index."""
    N, d, K = 20, 32, 9
    V = np.zeros((N, d), np.float16)
    V[np.arange(N), np.arange(N)] = 1.0
    idx, order, _ = oracle.select_one(V, K, None, None)
    assert np.array_equal(order, np.arange(K)) and np.array_equal(idx, np.arange(K))


def test_duplicate_of_a_kept_token_is_picked_last():
    N, d = 10, 16
    V = np.zeros((N, d), np.float16)
    V[np.arange(N - 1), np.arange(N - 1)] = 1.0
    V[N - 1] = V[0]
    idx, order, _ = oracle.select_one(V, N, None, None)
    assert order[-1] == N - 1 and np.array_equal(idx, np.arange(N))


def test_pure_saliency_is_top_k():
    rng = np.random.default_rng(11)
    N, d, K = 50, 16, 12
    V = rng.standard_normal((N, d)).astype(np.float16)
    A = rng.random(N).astype(np.float32)
    A[7] = A[3]  # a tie: the lower index must win
    idx, _, stage = oracle.select_one(V, K, None, A, alpha_pm=0, beta_pm=1000)
    assert (stage == -1).all()
    ref = sorted(range(N), key=lambda i: (-A[i], i))[:K]
    assert np.array_equal(idx, np.sort(ref))


def test_pure_query_single_concept_is_top_k_of_cosine():
    rng = np.random.default_rng(12)
    N, d, K = 60, 32, 10
    V = rng.standard_normal((N, d)).astype(np.float16)
    Q = (V[5:6].astype(np.float32) + 0.3 * rng.standard_normal((1, d))).astype(np.float16)
    idx, order, stage = oracle.select_one(V, K, Q, None, alpha_pm=1000, beta_pm=0)
    assert (stage == 1).all()
    score = _cos64(_deq(Q), _deq(V))[0]
    thr = np.sort(score)[::-1][K - 1]
    assert np.all(score[idx] >= thr - TOL)
    assert order[0] == 5


def test_budget_equal_to_n_keeps_everything():
    w = wl.Workload("t", B=1, N=24, d=32, K=24, T=0, J=3, seed=4, heavy_tail=False, linears=())
    x = wl.selector_inputs(w)
    idx, _, _ = oracle.select_one(x.V[0], 24, x.Q[0], x.A[0])
    assert np.array_equal(idx, np.arange(24))


def test_batch_equals_per_image():
    w = wl.Workload("t", B=3, N=40, d=64, K=10, T=0, J=3, seed=5, heavy_tail=False, linears=())
    x = wl.selector_inputs(w)
    got = oracle.select_batch(x.V, 10, x.Q, x.A)
    for b in range(3):
        assert np.array_equal(got[b], oracle.select_one(x.V[b], 10, x.Q[b], x.A[b])[0])


def test_gather_keeps_fp16_originals_then_text():
    w = wl.Workload("t", B=2, N=30, d=16, K=5, T=3, J=3, seed=6, heavy_tail=False, linears=())
    x = wl.selector_inputs(w)
    idx = oracle.select_batch(x.V, 5, x.Q, x.A)
    X = oracle.gather(x.V, idx, x.text)
    for b in range(2):
        assert np.array_equal(X[b, :5], x.V[b, idx[b]].astype(np.float32))
        assert np.array_equal(X[b, 5:], x.text[b].astype(np.float32))


def test_planted_diversity_mistake_is_caught():
    """Picking argmax instead of argmin of the max-cosine violates the stage-3 property."""
    w = wl.Workload("t", B=1, N=40, d=32, K=12, T=0, J=3, seed=8, heavy_tail=False, linears=())
    x = wl.selector_inputs(w)
    V = x.V[0]
    G = _cos64(_deq(V), _deq(V))
    kept = [0]
    m = G[:, 0].copy()
    m[0] = -np.inf
    picked = []
    for _ in range(5):
        cand = [i for i in range(40) if i not in kept]
        p = max(cand, key=lambda i: m[i])   # planted: argmax
        picked.append(p)
        kept.append(p)
        m = np.maximum(m, G[:, p])
    # the honest property check rejects at least one of these picks
    kept2 = [0]
    bad = False
    for p in picked:
        rest = [i for i in range(40) if i not in kept2]
        mm = G[np.ix_(rest, kept2)].max(axis=1)
        if G[p, kept2].max() > mm.min() + TOL:
            bad = True
        kept2.append(p)
    assert bad
