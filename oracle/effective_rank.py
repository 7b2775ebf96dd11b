"""Effective-rank head score and group-level classification.

TEST INFRASTRUCTURE ONLY (see the package docstring). Parity status: pinned
by ``tests/test_oracle_effective_rank.py`` (closed forms: rank one gives 1,
r equal singular values give r; three independent routes agree; the
classification budget reproduces the paper's retrieval counts).

Sec. 4 defines, for query head h with projections W_Q^h, W_K^h of shape
[d_head, d_model]:
  Eq. 2   M_h = W_K^T W_Q                        (d_model x d_model)
  Eq. 4   sigma_hat_k = sigma_k / sum_j sigma_j over the nonzero singular
          values of M_h, and ER(h) = exp(-sum_k sigma_hat_k log sigma_hat_k)
  Eq. 5-6 C_h = (W_Q W_Q^T)(W_K W_K^T) (d_head x d_head) has eigenvalues
          sigma_k(M_h)^2, so sigma_k = sqrt(lambda_k(C_h)).
Algorithm 1 clamps the eigenvalues at zero before the square root, sorts
heads by ER ascending and labels the lowest-k retrieval. The GQA extension
appendix averages the ER of a group's query heads and labels whole KV groups.
"""

import numpy as np

from .kv_memory import retrieval_groups


def effective_rank(sigma):
    """Eq. 4 on a vector of singular values; zero entries contribute nothing."""
    sigma = np.asarray(sigma, dtype=np.float64)
    sigma = sigma[sigma > 0.0]
    if sigma.size == 0:
        raise ValueError("effective rank of a zero matrix is undefined")
    p = sigma / sigma.sum()
    return float(np.exp(-np.sum(p * np.log(p))))


def kernel_attention_matrix(Wq_h, Wk_h):
    """Eq. 2: M_h = W_K^{h T} W_Q^h, a d_model x d_model matrix."""
    return np.asarray(Wk_h, dtype=np.float64).T @ np.asarray(Wq_h, dtype=np.float64)


def sigma_explicit(Wq_h, Wk_h):
    """Nonzero singular values of the explicitly built M_h.

    Values at or below the usual numerical-rank threshold
    (sigma_max * d_model * eps) are the zeros of a rank <= d_head matrix and
    are dropped, as Eq. 4 sums over nonzero values only.
    """
    M = kernel_attention_matrix(Wq_h, Wk_h)
    s = np.linalg.svd(M, compute_uv=False)
    tol = s.max() * max(M.shape) * np.finfo(np.float64).eps
    return s[s > tol]


def sigma_proxy(Wq_h, Wk_h):
    """Eq. 5-6 and Algorithm 1: sqrt(max(eig(C_h), 0)), C_h = (W_Q W_Q^T)(W_K W_K^T).

    C_h is a product of two symmetric PSD matrices and need not be symmetric,
    so a general eigen-solver is used and the real parts are kept.
    """
    Wq = np.asarray(Wq_h, dtype=np.float64)
    Wk = np.asarray(Wk_h, dtype=np.float64)
    C = (Wq @ Wq.T) @ (Wk @ Wk.T)
    lam = np.real(np.linalg.eigvals(C))
    return np.sqrt(np.maximum(lam, 0.0))


def sigma_qr(Wq_h, Wk_h):
    """Singular values of M_h through thin QR factors (a third, independent route).

    With W_Q^T = Q_q R_q and W_K^T = Q_k R_k (orthonormal columns),
    M_h = Q_k (R_k R_q^T) Q_q^T, so M_h and R_k R_q^T share their singular
    values.
    """
    _, Rq = np.linalg.qr(np.asarray(Wq_h, dtype=np.float64).T)
    _, Rk = np.linalg.qr(np.asarray(Wk_h, dtype=np.float64).T)
    return np.linalg.svd(Rk @ Rq.T, compute_uv=False)


def er_explicit(Wq_h, Wk_h):
    return effective_rank(sigma_explicit(Wq_h, Wk_h))


def er_proxy(Wq_h, Wk_h):
    return effective_rank(sigma_proxy(Wq_h, Wk_h))


def er_qr(Wq_h, Wk_h):
    s = sigma_qr(Wq_h, Wk_h)
    tol = s.max() * max(np.shape(Wq_h)) * np.finfo(np.float64).eps
    return effective_rank(s[s > tol])


def head_scores(Wq, Wk, n_kv_heads):
    """ER of every query head of one layer.

    Wq [Hq, d_head, d_model]; Wk [Hkv, d_head, d_model]. Query head h uses its
    own W_Q^h and the key projection of its group, h // (Hq // Hkv).
    """
    Hq = Wq.shape[0]
    g = Hq // n_kv_heads
    return np.array([er_proxy(Wq[h], Wk[h // g]) for h in range(Hq)])


def classify_groups(er_q_heads, n_kv_groups, sparsity_pct):
    """Group-level labels of Algorithm 1 with the GQA extension.

    Group score = mean ER of its member query heads (contiguous grouping);
    groups are sorted ascending with a stable sort, so ties go to the lower
    group index, and exactly k = ceil((1 - s) * G) lowest groups are labelled
    retrieval (0); the rest streaming (1).
    """
    er = np.asarray(er_q_heads, dtype=np.float64)
    H = er.shape[0]
    if H % n_kv_groups:
        raise ValueError("query heads must split evenly into KV groups")
    score = er.reshape(n_kv_groups, H // n_kv_groups).mean(axis=1)
    order = np.argsort(score, kind="stable")
    k = retrieval_groups(n_kv_groups, sparsity_pct)
    labels = np.ones(n_kv_groups, dtype=np.uint8)
    labels[order[:k]] = 0
    return labels
