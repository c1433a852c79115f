"""The timeline summary of the persistent kernel (host logic on a synthetic trace, no GPU)."""
import numpy as np
import pytest

from paper_2609_26100_gb300 import trace as T


def _synthetic(n_ctas=3, n_act=2, slots=T.ATTN_BASE + 2 * T.MAX_LAYERS + 16, t0=10_000_000):
    tr = np.zeros((n_ctas, slots), dtype=np.uint64)
    for c in range(n_ctas):
        for pi in range(4 * n_act + 1):
            for r in range(4):
                tr[c, pi * 8 + 2 * r] = t0 + 1000 * (10 * pi + r) + 100 * c      # first
                tr[c, pi * 8 + 2 * r + 1] = t0 + 1000 * (10 * pi + r + 5) + 100 * c  # last
        for j in range(n_act):
            tr[c, T.ATTN_BASE + 2 * j] = t0 + 1000 * (40 * j + 7)
            tr[c, T.ATTN_BASE + 2 * j + 1] = t0 + 1000 * (40 * j + 9)
    return tr.ravel()


def test_windows_layers_and_attention():
    s = T.summarize(_synthetic(), n_ctas=3, n_act=2)
    assert [(p["phase"], p["slot"]) for p in s["phases"]] == [
        ("qkv", 0), ("o", 0), ("gate_up", 0), ("down", 0), ("qkv", 1), ("o", 1), ("gate_up", 1), ("down", 1),
        ("lm_head", 2)]
    w = s["phases"][1]["mma"]  # pi = 1, role 2: first 10*1 + 2 = 12 ms-units, last +5, three CTAs
    assert w == {"first_min": 12.0, "first_median": 12.1, "last_max": 17.2, "ctas": 3}
    assert s["layers"][0] == {"slot": 0, "start": 0.0, "end": 38.2, "span_us": 38.2}
    assert s["attention"][1]["window"]["first_min"] == 47.0
    assert s["total_us"] == pytest.approx(88.2)


def test_missing_roles_and_empty_trace():
    tr = _synthetic().reshape(3, -1)
    tr[:, 8 * 2 + 2 * 1] = 0  # no B-operand activity in phase 2
    s = T.summarize(tr.ravel(), 3, 2)
    assert s["phases"][2]["b_operand"] is None
    empty = T.summarize(np.zeros(3 * (T.ATTN_BASE + 2 * T.MAX_LAYERS)), 3, 2)
    assert empty["phases"] == [] and empty["total_us"] == 0.0
    with pytest.raises(ValueError):
        T.summarize(np.zeros(30), 3, 2)
