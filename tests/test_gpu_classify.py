"""GPU head classifier (aoh_classify; Sec. 4, Eq. 2-6, Algorithm 1, GQA
appendix) against the oracle on the same bf16 weights.

ER values are compared with the oracle's head_scores (the Eq. 5-6 route,
float64). Labels are index work decided by floating point, so they are
checked exactly against the oracle's ranking applied to the GPU's own ER
values; where the score gaps are wide they must also equal the oracle's
labels from its own ER. Closed forms use weights that are exact in bf16.
"""

import math

import numpy as np
import pytest
import torch

from gpu_cases import ensure_lib
from oracle import effective_rank as oer
from paper_2608_06849_gb300 import aoh

pytestmark = pytest.mark.gpu


def _dev(a):
    """float64 numpy array whose values are exact in bf16 -> bf16 CUDA tensor."""
    t = torch.from_numpy(np.ascontiguousarray(a, dtype=np.float64)).to(torch.bfloat16)
    assert np.array_equal(t.double().numpy(), a), "construction is not exact in bf16"
    return t.cuda()


def _bf16(a):
    return torch.from_numpy(np.asarray(a, dtype=np.float64)).to(torch.bfloat16).double().numpy()


def _classify(wq, wk, sparsity):
    ensure_lib()
    Hkv = wk.shape[0]
    labels, er = aoh.aoh_classify(_dev(wq), _dev(wk), Hkv, sparsity)
    return np.array(labels), np.array(er)


def _check_labels(labels, er_gpu, er_oracle, Hkv, sparsity, gap=1e-6):
    assert labels.tolist() == oer.classify_groups(er_gpu, Hkv, sparsity).tolist()
    g = er_gpu.shape[0] // Hkv
    s = np.sort(er_oracle.reshape(Hkv, g).mean(axis=1))
    if np.all(np.diff(s) > gap * s[-1]):
        assert labels.tolist() == oer.classify_groups(er_oracle, Hkv, sparsity).tolist()


@pytest.mark.parametrize("dh,dm", [(128, 512), (64, 384), (128, 130)])
def test_random_weights_match_oracle(dh, dm):
    rng = np.random.default_rng(dh + dm)
    Hq, Hkv = 8, 2
    wq = _bf16(rng.standard_normal((Hq, dh, dm)) * rng.uniform(0.3, 3.0, size=(Hq, dh, 1)))
    wk = _bf16(rng.standard_normal((Hkv, dh, dm)) * rng.uniform(0.3, 3.0, size=(Hkv, dh, 1)))
    labels, er = _classify(wq, wk, 50)
    want = oer.head_scores(wq, wk, Hkv)
    np.testing.assert_allclose(er, want, rtol=1e-9)
    _check_labels(labels, er, want, Hkv, 50)


def test_qwen25_7b_layer_shape():
    """28 query / 4 KV heads, d_head 128, d_model 3584; spectra of varied decay."""
    rng = np.random.default_rng(7)
    Hq, Hkv, dh, dm = 28, 4, 128, 3584
    decay = np.geomspace(1.0, 1e-2, dh)
    wq = np.empty((Hq, dh, dm))
    for h in range(Hq):
        e = rng.uniform(0.0, 1.5)
        wq[h] = (decay ** e)[:, None] * rng.standard_normal((dh, dm))
    wk = rng.standard_normal((Hkv, dh, dm)) * (decay ** 0.5)[None, :, None]
    wq, wk = _bf16(wq), _bf16(wk)
    want = oer.head_scores(wq, wk, Hkv)
    for sparsity in (25, 50, 75):
        labels, er = _classify(wq, wk, sparsity)
        np.testing.assert_allclose(er, want, rtol=1e-9)
        _check_labels(labels, er, want, Hkv, sparsity)


@pytest.mark.parametrize("dh", [64, 128])
def test_closed_forms(dh):
    """Rank one gives 1; identity blocks give d_head; r equal singular values
    give r; singular values (3, 1) give exp of their entropy."""
    rng = np.random.default_rng(dh)
    dm = 2 * dh + 32
    eye = np.zeros((dh, dm))
    eye[:, :dh] = np.eye(dh)
    wq = np.zeros((4, dh, dm))
    v = _bf16(rng.standard_normal(dm))
    u = 2.0 ** -(np.arange(dh) % 5)
    wq[0] = u[:, None] * v[None, :]               # W_Q = u v^T: rank one
    wq[1] = eye                                   # identity block
    r = 5
    wq[2, :r, :r] = 1.75 * np.eye(r)              # r equal singular values
    wq[3, 0, 0], wq[3, 1, 1] = 3.0, 1.0           # singular values (3, 1)
    wk = eye[None]
    labels, er = _classify(wq, wk, 0)
    assert abs(er[0] - 1.0) < 1e-9
    assert abs(er[1] - dh) < 1e-9 * dh
    assert abs(er[2] - r) < 1e-9 * r
    two = math.exp(-(0.75 * math.log(0.75) + 0.25 * math.log(0.25)))
    assert abs(er[3] - two) < 1e-12
    assert labels.tolist() == [0]


def test_concentrated_heads_are_retrieval():
    """Groups whose heads have concentrated spectra are the ones labelled
    retrieval (the paper's premise, on constructed heads)."""
    rng = np.random.default_rng(5)
    dh, dm, Hkv, g = 128, 512, 4, 3
    wk = _bf16(rng.standard_normal((Hkv, dh, dm)))
    wq = np.empty((Hkv * g, dh, dm))
    concentrated = {1, 3}
    for kv in range(Hkv):
        for m in range(g):
            sig = np.geomspace(1.0, 1e-3, dh) if kv in concentrated else np.ones(dh)
            wq[kv * g + m] = sig[:, None] * rng.standard_normal((dh, dm))
    wq = _bf16(wq)
    labels, er = _classify(wq, wk, 50)
    assert labels.tolist() == [1, 0, 1, 0]
    np.testing.assert_allclose(er, oer.head_scores(wq, wk, Hkv), rtol=1e-9)


def test_budget_edges_and_ties():
    """0% sparsity labels every group retrieval, 100% none. Scaling W_Q by a
    power of two leaves ER bit-identical, so four groups built that way tie
    exactly and the stable rule picks the lowest index."""
    rng = np.random.default_rng(9)
    dh, dm, Hkv, g = 64, 256, 4, 2
    base_q = _bf16(rng.standard_normal((g, dh, dm)))
    base_k = _bf16(rng.standard_normal((dh, dm)))
    wq = np.concatenate([base_q * s for s in (1.0, 2.0, 1.0, 4.0)])
    wk = np.stack([base_k] * Hkv)
    lab0, er = _classify(wq, wk, 0)
    assert lab0.tolist() == [0, 0, 0, 0]
    lab100, _ = _classify(wq, wk, 100)
    assert lab100.tolist() == [1, 1, 1, 1]
    for kv in range(1, Hkv):
        assert er[kv * g] == er[0] and er[kv * g + 1] == er[1]
    lab75, er75 = _classify(wq, wk, 75)
    assert lab75.tolist() == oer.classify_groups(er75, Hkv, 75).tolist() == [0, 1, 1, 1]


def test_layers_in_one_call():
    """Several layers in one call give each layer's own result (labels by
    layer, ER within 1e-12 of the one-layer calls, whose d_model split, and
    so summation order, may differ) and agree with the oracle."""
    ensure_lib()
    rng = np.random.default_rng(13)
    L, Hq, Hkv, dh, dm = 3, 8, 2, 128, 256
    wq = _bf16(rng.standard_normal((L, Hq, dh, dm)) * rng.uniform(0.2, 2.0, size=(L, Hq, dh, 1)))
    wk = _bf16(rng.standard_normal((L, Hkv, dh, dm)))
    labels, ers = aoh.aoh_classify(_dev(wq), _dev(wk), Hkv, 50)
    assert len(labels) == L and len(ers) == L
    for l in range(L):
        lab1, er1 = _classify(wq[l], wk[l], 50)
        np.testing.assert_allclose(ers[l], er1, rtol=1e-12)
        want = oer.head_scores(wq[l], wk[l], Hkv)
        np.testing.assert_allclose(ers[l], want, rtol=1e-9)
        _check_labels(np.array(labels[l]), np.array(ers[l]), want, Hkv, 50)
