"""Pins of the H2Share oracle (the paper's H2Share section, Eq. sim, and the
GQA extension appendix)."""

import math

import numpy as np
import pytest

from oracle import attention as att
from oracle import h2share as hs


def _explicit_similarity(Wq_a, Wk_a, Wq_r, Wk_r):
    """Eq. sim from the explicit d_model x d_model kernel matrices."""
    Ma, Mr = Wk_a.T @ Wq_a, Wk_r.T @ Wq_r
    return float(np.sum(Ma * Mr) / (np.linalg.norm(Ma) * np.linalg.norm(Mr)))


def test_similarity_trace_route_matches_explicit_matrices():
    rng = np.random.default_rng(0)
    for dh, dm in [(4, 16), (8, 40), (3, 9)]:
        for _ in range(5):
            W = [rng.standard_normal((dh, dm)) * rng.uniform(0.2, 3, size=(dh, 1)) for _ in range(4)]
            got = hs.head_similarity(*W)
            assert abs(got - _explicit_similarity(*W)) < 1e-12


def test_similarity_closed_forms():
    rng = np.random.default_rng(1)
    Wq, Wk = rng.standard_normal((6, 30)), rng.standard_normal((6, 30))
    assert abs(hs.head_similarity(Wq, Wk, Wq, Wk) - 1.0) < 1e-13
    assert abs(hs.head_similarity(Wq, Wk, 3.0 * Wq, 0.5 * Wk) - 1.0) < 1e-13
    assert abs(hs.head_similarity(Wq, Wk, -Wq, Wk) + 1.0) < 1e-13
    Wq2, Wk2 = rng.standard_normal((6, 30)), rng.standard_normal((6, 30))
    assert abs(hs.head_similarity(Wq, Wk, Wq2, Wk2) - hs.head_similarity(Wq2, Wk2, Wq, Wk)) < 1e-13
    # kernel matrices on orthogonal subspaces of the model space: similarity 0
    Z = np.zeros((6, 30))
    A, B = Z.copy(), Z.copy()
    A[:, :6] = np.eye(6)
    B[:, 6:12] = np.eye(6)
    assert abs(hs.head_similarity(A, A, B, B)) < 1e-15


def test_group_similarity_is_the_mean_of_head_pairs():
    rng = np.random.default_rng(2)
    Hq, Hkv, dh, dm = 6, 3, 4, 20
    Wq_a, Wk_a = rng.standard_normal((Hq, dh, dm)), rng.standard_normal((Hkv, dh, dm))
    Wq_r, Wk_r = rng.standard_normal((Hq, dh, dm)), rng.standard_normal((Hkv, dh, dm))
    sim = hs.group_similarity(Wq_a, Wk_a, Wq_r, Wk_r)
    g = Hq // Hkv
    for ga in range(Hkv):
        for gr in range(Hkv):
            tot = 0.0
            for i in range(g):
                for j in range(g):
                    tot += _explicit_similarity(Wq_a[ga * g + i], Wk_a[ga], Wq_r[gr * g + j], Wk_r[gr])
            assert abs(sim[ga, gr] - tot / (g * g)) < 1e-12


def test_mapping_recovers_a_permuted_layer():
    rng = np.random.default_rng(3)
    Hq, Hkv, dh, dm = 8, 4, 4, 24
    Wq, Wk = rng.standard_normal((Hq, dh, dm)), rng.standard_normal((Hkv, dh, dm))
    perm = [2, 0, 3, 1]                       # reuse group r is anchor group perm[r]
    g = Hq // Hkv
    Wq_r = np.concatenate([Wq[p * g:(p + 1) * g] for p in perm])
    Wk_r = Wk[perm]
    sim = hs.group_similarity(Wq, Wk, Wq_r, Wk_r)
    assert hs.group_mapping(sim, [0, 0, 0, 0], [0, 0, 0, 0]).tolist() == perm
    # streaming reuse groups get -1; only retrieval anchors are candidates
    got = hs.group_mapping(sim, [0, 1, 0, 1], [0, 0, 1, 0])
    assert got[2] == -1
    assert all(a in (0, 2) for a in got[[0, 1, 3]])
    # ties go to the lower anchor index
    assert hs.group_mapping(np.ones((3, 2)), [1, 0, 0], [0, 0]).tolist() == [1, 1]


def test_importance_brute_force_and_invariants():
    rng = np.random.default_rng(4)
    g, d, T = 3, 8, 23
    q, k = rng.standard_normal((g, d)), rng.standard_normal((T, d)) * 2
    got = hs.group_importance(q, k)
    want = np.zeros(T)
    for h in range(g):
        sc = [sum(q[h, e] * k[j, e] for e in range(d)) / math.sqrt(d) for j in range(T)]
        mx = max(sc)
        ws = [math.exp(s - mx) for s in sc]
        tot = sum(ws)
        for j in range(T):
            want[j] += ws[j] / tot
    np.testing.assert_allclose(got, want, rtol=0, atol=1e-14)
    assert abs(got.sum() - g) < 1e-12


def test_topk_selection():
    imp = np.array([0.1, 0.5, 0.3, 0.5, 0.05, 0.3, 0.9])
    assert hs.select_topk(imp, 3).tolist() == [1, 3, 6]
    assert hs.select_topk(imp, 4).tolist() == [1, 2, 3, 6]          # tie 0.3: lower position
    assert hs.select_topk(imp, 100).tolist() == list(range(7))       # k >= n: every position
    rng = np.random.default_rng(5)
    x = rng.standard_normal(200)
    for k in (1, 17, 64, 199):
        sel = hs.select_topk(x, k)
        assert len(sel) == k and np.all(np.diff(sel) > 0)
        rest = np.setdiff1d(np.arange(200), sel)
        assert x[sel].min() >= x[rest].max()


def test_sparse_attention_special_cases():
    rng = np.random.default_rng(6)
    g, d, T, S, W = 2, 8, 30, 2, 5
    q = rng.standard_normal((g, d))
    k = rng.standard_normal((T, 1, d))
    v = rng.standard_normal((T, 1, d))
    full = att.decode_step(q, k, v, [0], S, W)                     # a retrieval group, position T-1
    np.testing.assert_allclose(hs.sparse_attend(q, k[:, 0], v[:, 0], np.arange(T)), full, rtol=0, atol=1e-14)
    one = hs.sparse_attend(q, k[:, 0], v[:, 0], [7])
    np.testing.assert_allclose(one, np.repeat(v[7], g, axis=0), rtol=0, atol=0)
    idx = [3, 11, 29, 0]
    a = hs.sparse_attend(q, k[:, 0], v[:, 0], idx)
    b = hs.sparse_attend(q, k[:, 0], v[:, 0], sorted(idx))
    np.testing.assert_allclose(a, b, rtol=0, atol=1e-15)
    # the selected positions of the full step's own importance carry most of its mass
    imp = hs.group_importance(q, k[:, 0])
    sel = hs.select_topk(imp, T)
    np.testing.assert_allclose(hs.sparse_attend(q, k[:, 0], v[:, 0], sel), full, rtol=0, atol=1e-14)
