"""H2Share: index-only cross-layer sparse attention (the paper's H2Share
section and its GQA extension appendix).

TEST INFRASTRUCTURE ONLY (see the package docstring). Parity status:
pinned by ``tests/test_oracle_h2share.py`` (brute force over explicit
d_model x d_model kernel matrices for the head similarity, a full softmax
for the selection, special cases that reduce to plain attention).

What the paper fixes:
  * layers form anchor-reuse blocks; an anchor layer's retrieval heads run
    full attention and select the top-k token positions by their attention
    scores; a reuse layer's retrieval heads attend only to their own K/V at
    the positions borrowed from the mapped anchor head (no K/V crosses
    layers); streaming heads keep their sink + window attention;
  * the mapping sends each reuse retrieval head to the anchor retrieval head
    whose kernel attention matrix is most similar under the normalised
    Frobenius inner product (Eq. sim), computed through traces of d_head x
    d_head products;
  * with GQA, similarities of the group pairs are the mean over their query
    head pairs, and all query heads of a group borrow one index set.

Readings taken where the paper is silent:
  * the importance of key j for an anchor retrieval group is the sum over
    the group's query heads of their attention probabilities at j (the
    softmax over all positions the head attends); the group keeps the
    min(k, t + 1) most important positions, ties to the lower position,
    listed in increasing order;
  * selection happens at every decode step, over the positions 0..t that
    the anchor step attends (its new token included);
  * a reuse retrieval group attends with plain softmax attention to its own
    K/V at exactly the borrowed positions;
  * the mapping argmax breaks ties toward the lower anchor group index.
"""

import numpy as np


def group_importance(q_group, k_seq):
    """Importance of every cached position for one retrieval KV group.

    q_group [g, d] (the group's query heads at the current step), k_seq
    [t+1, d] (the group's keys at positions 0..t). Returns [t+1]: the sum
    over the g heads of softmax(q k^T / sqrt(d)).
    """
    q = np.asarray(q_group, dtype=np.float64)
    k = np.asarray(k_seq, dtype=np.float64)
    s = (q @ k.T) / np.sqrt(q.shape[1])
    s = s - s.max(axis=1, keepdims=True)
    p = np.exp(s)
    p = p / p.sum(axis=1, keepdims=True)
    return p.sum(axis=0)


def select_topk(importance, k):
    """The min(k, n) most important positions, ties to the lower position,
    in increasing order."""
    imp = np.asarray(importance, dtype=np.float64)
    n = imp.shape[0]
    order = sorted(range(n), key=lambda j: (-imp[j], j))
    return np.array(sorted(order[:min(k, n)]), dtype=np.int64)


def sparse_attend(q_group, k_seq, v_seq, idx):
    """Softmax attention of the group's query heads over the positions idx of
    their own keys and values. q_group [g, d], k_seq / v_seq [T, d]."""
    q = np.asarray(q_group, dtype=np.float64)
    k = np.asarray(k_seq, dtype=np.float64)[np.asarray(idx)]
    v = np.asarray(v_seq, dtype=np.float64)[np.asarray(idx)]
    s = (q @ k.T) / np.sqrt(q.shape[1])
    s = s - s.max(axis=1, keepdims=True)
    p = np.exp(s)
    p = p / p.sum(axis=1, keepdims=True)
    return p @ v


def head_similarity(Wq_a, Wk_a, Wq_r, Wk_r):
    """Eq. sim for one anchor head (Wq_a, Wk_a: [d_head, d_model]) and one
    reuse head: <M_a, M_r>_F / (|M_a|_F |M_r|_F), M = W_K^T W_Q, through
    the trace identities (everything is d_head x d_head)."""
    Wq_a, Wk_a = np.asarray(Wq_a, np.float64), np.asarray(Wk_a, np.float64)
    Wq_r, Wk_r = np.asarray(Wq_r, np.float64), np.asarray(Wk_r, np.float64)
    num = np.trace((Wq_a @ Wq_r.T) @ (Wk_r @ Wk_a.T))
    na = np.trace((Wq_a @ Wq_a.T) @ (Wk_a @ Wk_a.T))
    nr = np.trace((Wq_r @ Wq_r.T) @ (Wk_r @ Wk_r.T))
    return num / np.sqrt(na * nr)


def group_similarity(Wq_a, Wk_a, Wq_r, Wk_r):
    """[G_a, G_r] group-pair similarities: the mean of Eq. sim over the
    query-head pairs of the two groups. Wq_* [Hq, d_head, d_model],
    Wk_* [Hkv, d_head, d_model]; query head h uses key group h // (Hq/Hkv)."""
    Hq, Hkv = Wq_a.shape[0], Wk_a.shape[0]
    g = Hq // Hkv
    out = np.zeros((Hkv, Hkv))
    for ga in range(Hkv):
        for gr in range(Hkv):
            vals = [head_similarity(Wq_a[ha], Wk_a[ga], Wq_r[hr], Wk_r[gr])
                    for ha in range(ga * g, (ga + 1) * g) for hr in range(gr * g, (gr + 1) * g)]
            out[ga, gr] = np.mean(vals)
    return out


def group_mapping(sim, anchor_labels, reuse_labels):
    """For every reuse retrieval group (label 0), the anchor retrieval group
    of highest similarity (ties to the lower index); -1 for streaming
    groups. sim [G_a, G_r] from ``group_similarity``."""
    sim = np.asarray(sim, dtype=np.float64)
    anchors = [a for a in range(sim.shape[0]) if int(anchor_labels[a]) == 0]
    out = np.full(sim.shape[1], -1, dtype=np.int64)
    for r in range(sim.shape[1]):
        if int(reuse_labels[r]) != 0 or not anchors:
            continue
        best = anchors[0]
        for a in anchors[1:]:
            if sim[a, r] > sim[best, r]:
                best = a
        out[r] = best
    return out
