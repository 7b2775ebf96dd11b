"""Mutation check of the oracle's pins.

A plausible mistake is planted in a copy of the oracle's source (never in the
oracle itself), the copy is loaded as a module, and at least one pin must
fail on it. This shows the pins would catch a dropped term, a wrong sign, an
off-by-one in the mask or a wrong operand.
"""

import os
import types

import pytest

import oracle_pins

SRC = os.path.join(os.path.dirname(os.path.dirname(os.path.abspath(__file__))), "oracle", "attention.py")

MUTANTS = {
    "window_off_by_one": ("(i - j < W)", "(i - j <= W)"),
    "sink_off_by_one": ("(j < S)", "(j <= S)"),
    "no_causal": ("causal = j <= i", "causal = j <= i + 1"),
    "scale_dropped": ("scale = 1.0 / np.sqrt(d)", "scale = 1.0"),
    "scale_wrong": ("scale = 1.0 / np.sqrt(d)", "scale = 1.0 / d"),
    "no_max_subtract_sign": ("p = np.exp(s - m)", "p = np.exp(m - s)"),
    "no_normalise": ("p = p / p.sum(axis=1, keepdims=True)", "p = p"),
    "kv_map_modulo": ("for h in range(kv * g, (kv + 1) * g):", "for h in [x for x in range(Hq) if x % Hkv == kv]:"),
    "labels_swapped": ("streaming = int(labels[kv]) == STREAMING", "streaming = int(labels[kv]) == RETRIEVAL"),
    "ring_slot_wrong_base": ("return S + (p - S) % W", "return S + p % W"),
    "value_uses_key": ("out[:, h, :] = p @ v[:, kv, :]", "out[:, h, :] = p @ k[:, kv, :]"),
    "decode_wrong_row": ("t = k_seq.shape[0] - 1", "t = k_seq.shape[0] - 2"),
    "chunk_window_off_by_one": ("(j >= (i // chunk) * chunk - W))", "(j > (i // chunk) * chunk - W))"),
    "chunk_per_query": ("(j >= (i // chunk) * chunk - W))", "(j >= i - W))"),
    "chunk_ignored": ("    if chunk:\n        return causal", "    if False:\n        return causal"),
    # the scalar form alone (the vector form, which prefill uses, untouched)
    "scalar_window_off_by_one": ("return j < S or i - j < W", "return j < S or i - j <= W"),
    "scalar_chunk_per_query": ("return j < S or j >= (i // chunk) * chunk - W", "return j < S or j >= i - W"),
    "scalar_not_causal": ("    if j > i:\n        return False", "    if j > i + 1:\n        return False"),
}


def _load_mutant(old, new):
    src = open(SRC).read()
    assert src.count(old) >= 1, old
    mod = types.ModuleType("oracle_attention_mutant")
    exec(compile(src.replace(old, new), "mutant", "exec"), mod.__dict__)
    return mod


@pytest.mark.parametrize("name", sorted(MUTANTS))
def test_pins_catch_mutant(name):
    old, new = MUTANTS[name]
    mod = _load_mutant(old, new)
    caught = []
    for pin in oracle_pins.ALL_PINS:
        try:
            pin(mod)
        except Exception:
            caught.append(pin.__name__)
    assert caught, f"no pin catches mutant {name}"


# ---- effective rank and KV bytes: plant the mistake in a copy of the oracle
# module, swap the copy in for the duration of the check, run the pin tests.

import importlib  # noqa: E402

import oracle  # noqa: E402

ER_MUTANTS = {
    "no_sqrt": ("return np.sqrt(np.maximum(lam, 0.0))", "return np.maximum(lam, 0.0)"),
    "log2": ("np.exp(-np.sum(p * np.log(p)))", "np.exp(-np.sum(p * np.log2(p)))"),
    "no_normalise": ("p = sigma / sigma.sum()", "p = sigma / sigma.max()"),
    "gram_wrong_side": ("C = (Wq @ Wq.T) @ (Wk @ Wk.T)", "C = (Wq @ Wk.T) @ (Wk @ Wq.T) * 0 + (Wq @ Wq.T)"),
    "m_transposed_operand": ("return np.asarray(Wk_h, dtype=np.float64).T @ np.asarray(Wq_h, dtype=np.float64)",
                             "return np.asarray(Wq_h, dtype=np.float64).T @ np.asarray(Wq_h, dtype=np.float64)"),
    "descending_sort": ('order = np.argsort(score, kind="stable")', 'order = np.argsort(-score, kind="stable")'),
    "max_not_mean": ("score = er.reshape(n_kv_groups, H // n_kv_groups).mean(axis=1)",
                     "score = er.reshape(n_kv_groups, H // n_kv_groups).max(axis=1)"),
}
KV_MUTANTS = {
    "floor_budget": ("return -(-num // 100)", "return num // 100"),
    "no_v": ("return batch * tokens * d_head * 2 * elem_bytes", "return batch * tokens * d_head * elem_bytes"),
    "window_only": ("n_streaming * (S + W)", "n_streaming * W"),
}


H2_MUTANTS = {
    "similarity_transposed_key_product": ("num = np.trace((Wq_a @ Wq_r.T) @ (Wk_r @ Wk_a.T))",
                                          "num = np.trace((Wq_a @ Wq_r.T) @ (Wk_a @ Wk_r.T))"),
    "similarity_no_norm": ("return num / np.sqrt(na * nr)", "return num / np.sqrt(na)"),
    "importance_unnormalised": ("p = p / p.sum(axis=1, keepdims=True)\n    return p.sum(axis=0)",
                                "return p.sum(axis=0)"),
    "topk_ties_high": ("key=lambda j: (-imp[j], j)", "key=lambda j: (-imp[j], -j)"),
    "sparse_no_scale": ("s = (q @ k.T) / np.sqrt(q.shape[1])\n    s = s - s.max(axis=1, keepdims=True)\n    p = np.exp(s)\n    p = p / p.sum(axis=1, keepdims=True)\n    return p @ v",
                        "s = (q @ k.T)\n    s = s - s.max(axis=1, keepdims=True)\n    p = np.exp(s)\n    p = p / p.sum(axis=1, keepdims=True)\n    return p @ v"),
    "mapping_ties_high": ("if sim[a, r] > sim[best, r]:", "if sim[a, r] >= sim[best, r]:"),
    "group_mean_max": ("out[ga, gr] = np.mean(vals)", "out[ga, gr] = np.max(vals)"),
}


def _mutated(modname, old, new):
    path = os.path.join(os.path.dirname(SRC), modname + ".py")
    src = open(path).read()
    assert src.count(old) >= 1, old
    mod = types.ModuleType("oracle." + modname)
    mod.__package__ = "oracle"
    exec(compile(src.replace(old, new), "mutant", "exec"), mod.__dict__)
    return mod


def _failures(test_module_name, monkeypatch, modname, mod):
    monkeypatch.setattr(oracle, modname, mod)
    tm = importlib.import_module(test_module_name)
    monkeypatch.setattr(tm, {"effective_rank": "er", "kv_memory": "kvm", "h2share": "hs"}[modname], mod)
    failed = 0
    for name in dir(tm):
        if not name.startswith("test_"):
            continue
        fn = getattr(tm, name)
        marks = getattr(fn, "pytestmark", [])
        params = [m for m in marks if m.name == "parametrize"]
        argsets = [{}]
        for m in params:
            argsets = [dict(a, **{m.args[0].split(",")[0]: v}) if "," not in m.args[0]
                       else dict(a, **dict(zip([x.strip() for x in m.args[0].split(",")], v)))
                       for a in argsets for v in m.args[1]]
        for kw in argsets:
            try:
                fn(**kw)
            except Exception:
                failed += 1
    return failed


@pytest.mark.parametrize("name", sorted(ER_MUTANTS))
def test_er_pins_catch_mutant(name, monkeypatch):
    mod = _mutated("effective_rank", *ER_MUTANTS[name])
    assert _failures("test_oracle_effective_rank", monkeypatch, "effective_rank", mod) > 0


@pytest.mark.parametrize("name", sorted(KV_MUTANTS))
def test_kv_pins_catch_mutant(name, monkeypatch):
    mod = _mutated("kv_memory", *KV_MUTANTS[name])
    assert _failures("test_oracle_kv_memory", monkeypatch, "kv_memory", mod) > 0


@pytest.mark.parametrize("name", sorted(H2_MUTANTS))
def test_h2share_pins_catch_mutant(name, monkeypatch):
    mod = _mutated("h2share", *H2_MUTANTS[name])
    assert _failures("test_oracle_h2share", monkeypatch, "h2share", mod) > 0
