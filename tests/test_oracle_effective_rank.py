"""Pins of the effective-rank oracle (Sec. 4, Eq. 2-6, Algorithm 1, GQA appendix)."""

import math

import numpy as np
import pytest

from oracle import effective_rank as er


def _orth(rng, n, k):
    q, _ = np.linalg.qr(rng.standard_normal((n, k)))
    return q[:, :k]


def _weights_with_sigma(rng, sigma, d_head, d_model):
    """W_Q, W_K ([d_head, d_model]) whose M = W_K^T W_Q has singular values sigma."""
    r = len(sigma)
    U = _orth(rng, d_model, d_head)  # key-side directions
    V = _orth(rng, d_model, d_head)  # query-side directions
    A = np.zeros((d_head, d_head))
    A[:r, :r] = np.diag(sigma)
    Wk = U.T                     # W_K^T = U
    Wq = A @ V.T                 # M = U A V^T
    return Wq, Wk


ROUTES = [er.er_explicit, er.er_qr]


@pytest.mark.parametrize("route", ROUTES + [er.er_proxy], ids=lambda f: f.__name__)
def test_rank_one_gives_one(route):
    rng = np.random.default_rng(0)
    Wq, Wk = _weights_with_sigma(rng, [2.5], 8, 40)
    tol = 1e-6 if route is er.er_proxy else 1e-12   # eig of C squares the conditioning
    assert abs(route(Wq, Wk) - 1.0) < tol


@pytest.mark.parametrize("route", ROUTES + [er.er_proxy], ids=lambda f: f.__name__)
@pytest.mark.parametrize("r", [2, 3, 8])
def test_equal_singular_values_give_their_count(route, r):
    rng = np.random.default_rng(r)
    Wq, Wk = _weights_with_sigma(rng, [1.7] * r, 8, 48)
    tol = 1e-6 if (route is er.er_proxy and r < 8) else 1e-10
    assert abs(route(Wq, Wk) - r) < tol * r


def test_identity_blocks_give_d_head():
    d_head, d_model = 8, 32
    W = np.zeros((d_head, d_model))
    W[:, :d_head] = np.eye(d_head)
    for route in ROUTES + [er.er_proxy]:
        assert abs(route(W, W) - d_head) < 1e-12


def test_two_value_closed_form():
    """sigma = (3, 1): p = (3/4, 1/4), ER = exp(-(3/4 ln 3/4 + 1/4 ln 1/4))."""
    rng = np.random.default_rng(7)
    Wq, Wk = _weights_with_sigma(rng, [3.0, 1.0], 4, 24)
    want = math.exp(-(0.75 * math.log(0.75) + 0.25 * math.log(0.25)))
    for route in ROUTES:
        assert abs(route(Wq, Wk) - want) < 1e-12
    assert abs(er.er_proxy(Wq, Wk) - want) < 1e-6


@pytest.mark.parametrize("d_model,d_head", [(32, 4), (96, 8), (64, 16)])
def test_three_routes_agree_on_random_weights(d_model, d_head):
    rng = np.random.default_rng(d_model + d_head)
    for _ in range(4):
        Wq = rng.standard_normal((d_head, d_model))
        Wk = rng.standard_normal((d_head, d_model)) * rng.uniform(0.2, 3.0, size=(d_head, 1))
        s1 = np.sort(er.sigma_explicit(Wq, Wk))[::-1]
        s2 = np.sort(er.sigma_proxy(Wq, Wk))[::-1]
        s3 = np.sort(er.sigma_qr(Wq, Wk))[::-1]
        assert s1.shape == (d_head,)
        np.testing.assert_allclose(s2, s1, rtol=1e-9)
        np.testing.assert_allclose(s3, s1, rtol=1e-9)
        a, b, c = er.er_explicit(Wq, Wk), er.er_proxy(Wq, Wk), er.er_qr(Wq, Wk)
        assert abs(b - a) < 1e-9 * a and abs(c - a) < 1e-9 * a
        assert 1.0 <= a <= d_head


def test_explicit_matrix_is_wk_transpose_wq():
    rng = np.random.default_rng(3)
    Wq = rng.standard_normal((4, 10))
    Wk = rng.standard_normal((4, 10))
    M = er.kernel_attention_matrix(Wq, Wk)
    x_ctx = rng.standard_normal((6, 10))
    x_i = rng.standard_normal(10)
    # Eq. 1: scores = X_ctx W_K^T W_Q x_i equals (X_ctx W_K^T)(W_Q x_i)
    np.testing.assert_allclose(x_ctx @ M @ x_i, (x_ctx @ Wk.T) @ (Wq @ x_i), rtol=1e-12)


def test_invariances():
    """ER ignores an overall scale and a rotation of the model space."""
    rng = np.random.default_rng(11)
    Wq = rng.standard_normal((8, 40))
    Wk = rng.standard_normal((8, 40))
    base = er.er_proxy(Wq, Wk)
    R = _orth(rng, 40, 40)
    assert abs(er.er_proxy(3.0 * Wq, Wk) - base) < 1e-9
    assert abs(er.er_proxy(Wq @ R, Wk @ R) - base) < 1e-9


def test_budget_formula():
    # k = ceil((1 - s) G): the paper's GQA models at 25/50/75 % sparsity
    assert [er.retrieval_groups(4, s) for s in (0, 25, 50, 75, 100)] == [4, 3, 2, 1, 0]
    assert [er.retrieval_groups(8, s) for s in (25, 50, 75)] == [6, 4, 2]
    assert er.retrieval_groups(7, 50) == 4  # ceil(3.5)
    assert er.retrieval_groups(3, 10) == 3  # ceil(2.7)


def test_classify_groups_mean_and_ties():
    # 8 query heads, 4 groups of 2; group means 2.0, 1.0, 2.0, 5.0
    er_q = np.array([1.0, 3.0, 0.5, 1.5, 2.5, 1.5, 4.0, 6.0])
    lab = er.classify_groups(er_q, 4, 50)
    # lowest two: group 1 (1.0), then the tie 0 vs 2 at 2.0 goes to group 0
    assert lab.tolist() == [0, 0, 1, 1]
    assert er.classify_groups(er_q, 4, 75).tolist() == [1, 0, 1, 1]
    assert er.classify_groups(er_q, 4, 0).tolist() == [0, 0, 0, 0]


def test_classification_end_to_end_on_constructed_heads():
    """Heads built with concentrated spectra are the ones labelled retrieval."""
    rng = np.random.default_rng(5)
    d_head, d_model, G, g = 8, 64, 4, 2
    Wk = np.zeros((G, d_head, d_model))
    Wq = np.zeros((G * g, d_head, d_model))
    concentrated = {1, 3}
    for kv in range(G):
        Wk[kv] = _orth(rng, d_model, d_head).T
        for m in range(g):
            h = kv * g + m
            sig = np.geomspace(1.0, 1e-3, d_head) if kv in concentrated else np.ones(d_head)
            V = _orth(rng, d_model, d_head)
            Wq[h] = np.diag(sig) @ V.T
    scores = er.head_scores(Wq, Wk, G)
    assert er.classify_groups(scores, G, 50).tolist() == [1, 0, 1, 0]
