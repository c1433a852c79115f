"""Pins of the CPU oracle against facts fixed outside it: published vectors, printed table values,
closed forms, library routines and brute force on tiny inputs (no GPU)."""
import math
import os

import numpy as np
import pytest
import torch

from oracle import philox, tss_oracle as O
from paper_2609_26100_gb300 import synth

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def _rows(name):
    with open(os.path.join(GOLDEN, name)) as f:
        return [ln.split() for ln in f if ln.strip() and not ln.startswith("#")]


# ---------------------------------------------------------------------------------------------
# Philox4x32-10 (the generator behind the sampling uniforms)
# ---------------------------------------------------------------------------------------------
def test_philox_known_answers():
    for row in _rows("philox4x32_10_kat.txt"):
        v = [int(x, 16) for x in row]
        out = philox.philox4x32_10(np.array(v[:4], np.uint64), np.array(v[4:6], np.uint64))
        assert [int(x) for x in out] == v[6:10]


def test_uniform24_is_exact_fp32_in_unit_interval():
    u = philox.verify_uniforms(seed=42, offset=7, req=3, n_slots=4096)
    assert np.all(u >= 0) and np.all(u < 1)
    assert np.array_equal(u.astype(np.float32).astype(np.float64), u)
    assert abs(u.mean() - 0.5) < 0.02
    # distinct counters give distinct streams
    assert not np.array_equal(u[:16], philox.verify_uniforms(42, 7, 4, 16))
    assert not np.array_equal(u[:16], philox.verify_uniforms(42, 8, 3, 16))


# ---------------------------------------------------------------------------------------------
# Number formats
# ---------------------------------------------------------------------------------------------
def test_round_to_bf16_ties_and_library_agreement():
    e = 2.0 ** -8
    x = np.array([1.0, 1 + e, 1 + 3 * e, -(1 + 3 * e), 3.0e-3, 65504.0], np.float32)
    want = np.array([1.0, 1.0, 1 + 4 * e, -(1 + 4 * e)], np.float32)
    assert np.array_equal(O.round_to_bf16(x)[:4], want)
    r = np.random.default_rng(0).standard_normal(100000).astype(np.float32) * 3
    lib = torch.from_numpy(r).to(torch.bfloat16).to(torch.float32).numpy()
    assert np.array_equal(O.round_to_bf16(r), lib)


def test_bf16_bits_roundtrip():
    t = synth.normal_bf16((1000,), 1, "t", 0.5)
    u16 = t.view(torch.int16).numpy().view(np.uint16)
    assert np.array_equal(O.bf16_bits_to_f32(u16), t.to(torch.float32).numpy())


# ---------------------------------------------------------------------------------------------
# LLaMA block pieces
# ---------------------------------------------------------------------------------------------
def test_rmsnorm_closed_forms():
    h = np.array([[3.0, 4.0]])
    out = O.rms_norm(h, np.array([1.0, 2.0]), 0.0)
    r = math.sqrt((9 + 16) / 2)
    assert np.allclose(out, [[3 / r, 8 / r]], rtol=0, atol=1e-15)
    c = np.full((1, 64), -2.5)
    g = np.linspace(0.5, 1.5, 64)
    assert np.allclose(O.rms_norm(c, g, 0.0), -g, atol=1e-15)
    # eps enters under the square root: a zero row stays zero, finite, and (3, 4) with eps = 0.5
    # divides by sqrt(12.5 + 0.5), not by sqrt(12.5) + 0.5
    assert np.all(O.rms_norm(np.zeros((1, 8)), np.ones(8), 1e-5) == 0)
    assert np.allclose(O.rms_norm(h, np.ones(2), 0.5), [[3 / math.sqrt(13.0), 4 / math.sqrt(13.0)]], rtol=0, atol=1e-15)


def test_rope_is_complex_rotation_of_half_pairs():
    rng = np.random.default_rng(1)
    n, H, D, theta = 7, 3, 16, 1e4
    x = rng.standard_normal((n, H, D))
    pos = np.array([0, 1, 2, 17, 1000, 4095, 16392])
    cos, sin = O.rope_cos_sin(pos, D, theta, np.float64)
    out = O.apply_rope(x, cos, sin)
    half = D // 2
    z = x[..., :half] + 1j * x[..., half:]
    w = np.array([[np.exp(1j * p * theta ** (-2.0 * i / D)) for i in range(half)] for p in pos])
    zr = z * w[:, None, :]
    assert np.allclose(out[..., :half], zr.real, atol=1e-12)
    assert np.allclose(out[..., half:], zr.imag, atol=1e-12)
    assert np.allclose(out[0], x[0], atol=0)  # position 0 is the identity


def test_rope_scores_depend_on_relative_position_only():
    rng = np.random.default_rng(2)
    D = 32
    q = rng.standard_normal((1, 1, D))
    k = rng.standard_normal((1, 1, D))
    vals = []
    for p in (0, 5, 333, 2047):
        cq, sq = O.rope_cos_sin([p], D, 1e4, np.float64)
        ck, sk = O.rope_cos_sin([p + 9], D, 1e4, np.float64)
        vals.append(float(np.sum(O.apply_rope(q, cq, sq) * O.apply_rope(k, ck, sk))))
    assert np.allclose(vals, vals[0], atol=1e-10)


def test_silu_closed_forms():
    assert O.silu(np.array([0.0]))[0] == 0.0
    assert abs(O.silu(np.array([1.0]))[0] - 1 / (1 + math.exp(-1))) < 1e-15
    assert abs(O.silu(np.array([30.0]))[0] - 30.0) < 1e-10


def _brute_attention(q, k_ctx, v_ctx, k_blk, v_blk, parents):
    N, H, D = q.shape
    out = np.zeros_like(q)
    for i in range(N):
        anc = []
        j = i
        while j != -1:
            anc.append(j)
            j = parents[j]
        for h in range(H):
            keys = [k_ctx[h, c] for c in range(k_ctx.shape[1])] + [k_blk[j, h] for j in anc]
            vals = [v_ctx[h, c] for c in range(v_ctx.shape[1])] + [v_blk[j, h] for j in anc]
            s = [float(np.dot(q[i, h], kk)) / math.sqrt(D) for kk in keys]
            m = max(s)
            e = [math.exp(x - m) for x in s]
            z = sum(e)
            out[i, h] = sum(w / z * vv for w, vv in zip(e, vals))
    return out


@pytest.mark.parametrize("parents", [[-1], [-1, 0, 1, 2], [-1, 0, 0, 1, 1, 2, 5]])
def test_block_attention_matches_brute_force(parents):
    rng = np.random.default_rng(len(parents))
    N, H, D, C = len(parents), 2, 8, 5
    q, kb, vb = (rng.standard_normal((N, H, D)) for _ in range(3))
    kc, vc = rng.standard_normal((H, C, D)), rng.standard_normal((H, C, D))
    got = O.block_attention(q, kc, vc, kb, vb, O.ancestor_or_self(parents))
    assert np.allclose(got, _brute_attention(q, kc, vc, kb, vb, parents), atol=1e-12)


def test_attention_without_context_returns_own_value():
    rng = np.random.default_rng(3)
    q, k, v = (rng.standard_normal((1, 2, 4)) for _ in range(3))
    e = np.zeros((2, 0, 4))
    assert np.array_equal(O.block_attention(q, e, e, k, v, np.ones((1, 1), bool)), v)


def _closed_form_model():
    """L=1, d=2, H=1, D=2, F=1, V=3 with hand-chosen, non-symmetric weights."""
    arch = synth.Arch(n_layers=1, d_model=2, n_heads=1, head_dim=2, d_mlp=1, vocab=3, rms_eps=0.0)
    w = {
        "embed": np.array([[3.0, 4.0], [1.0, 0.0], [0.0, 1.0]]),
        "lm_head": np.array([[1.0, 0.0], [0.0, 1.0], [1.0, 1.0]]),
        "final_norm": np.array([1.0, 0.5]),
        "layers": [{
            "attn_norm": np.array([1.0, 1.0]),
            "wq": np.array([[0.3, -1.0], [2.0, 0.1]]),
            "wk": np.array([[1.0, 0.0], [0.5, 1.0]]),
            "wv": np.array([[1.0, 2.0], [0.0, 1.0]]),
            "wo": np.array([[0.0, 1.0], [2.0, 0.0]]),
            "mlp_norm": np.array([1.0, 1.0]),
            "w_gate": np.array([[1.0, 0.0]]),
            "w_up": np.array([[0.0, 1.0]]),
            "w_down": np.array([[1.0], [2.0]]),
        }],
    }
    return arch, w


def test_single_token_block_closed_form():
    arch, w = _closed_form_model()
    kv = [O.empty_kv(arch, np.float64)]
    logits, new_kv, hid = O.verify_request(w, arch, frozenset(), [0], [-1], 0, kv, np.float64,
                                           return_hidden=True)
    # Hand evaluation: h0 = (3, 4); xn = h0 / sqrt(12.5); one key, so the attention output is v.
    r0 = math.sqrt(12.5)
    x0, x1 = 3 / r0, 4 / r0
    v0, v1 = x0 + 2 * x1, x1
    v0, v1 = (float(O.round_to_bf16(np.array([v0]))[0]), float(O.round_to_bf16(np.array([v1]))[0]))
    h1 = (3 + v1, 4 + 2 * v0)  # wo = [[0, 1], [2, 0]]
    r1 = math.sqrt((h1[0] ** 2 + h1[1] ** 2) / 2)
    y0, y1 = h1[0] / r1, h1[1] / r1
    m = y0 / (1 + math.exp(-y0)) * y1  # silu(gate) * up
    h2 = (h1[0] + m, h1[1] + 2 * m)
    r2 = math.sqrt((h2[0] ** 2 + h2[1] ** 2) / 2)
    f0, f1 = h2[0] / r2, 0.5 * h2[1] / r2
    assert np.allclose(hid[0], h2, atol=1e-13)
    assert np.allclose(logits[0], [f0, f1, f0 + f1], atol=1e-13)


# ---------------------------------------------------------------------------------------------
# Controller (Sec. "Domain-Aware Skip Controller", Sec. "Domain-to-Configuration Mapping")
# ---------------------------------------------------------------------------------------------
def test_sparsity_ratio_reproduces_table1():
    for L, _domain, pct, layers in _rows("table1_skip_sets.txt"):
        S = [int(x) for x in layers.split(",")]
        assert round(100 * O.sparsity_ratio(S, int(L)), 1) == float(pct)


def test_unknown_domain_falls_back_to_dense():
    phi = {0: [3, 25, 30], 4: [1]}
    assert O.skip_set(phi, 0) == frozenset({3, 25, 30})
    assert O.skip_set(phi, 1) == frozenset()
    assert O.skip_set(phi, -7) == frozenset()
    assert O.mask_to_set(O.set_to_mask({0, 5, 63})) == frozenset({0, 5, 63})


def test_union_and_row_lists_brute_force():
    rng = np.random.default_rng(5)
    L = 12
    for _ in range(50):
        B = rng.integers(1, 6)
        skips = [frozenset(np.flatnonzero(rng.random(L) < 0.4).tolist()) for _ in range(B)]
        nodes = rng.integers(1, 5, B).tolist()
        rows = O.layer_row_lists(skips, nodes, L)
        assert sorted(rows) == O.union_active_layers(skips, L)
        for l in range(L):
            brute = [r for b in range(B) for r in range(sum(nodes[:b]), sum(nodes[:b + 1])) if l not in skips[b]]
            assert rows.get(l, []) == brute


# ---------------------------------------------------------------------------------------------
# Greedy decision rules
# ---------------------------------------------------------------------------------------------
def test_argmax_ties_and_margin():
    assert O.argmax_lowest([0.5, 1.0, 1.0]) == 1
    assert O.top2_margin([1.0, 1.0, 0.0]) == 0.0
    assert O.top2_margin([0.0, 2.0, 0.5]) == 1.5


def test_tree_accept_equals_longest_matching_root_path():
    rng = np.random.default_rng(6)
    parents = synth.eagle_tree(20, (3, 2, 2, 1))
    ch = O.children_of(parents)
    leaves = [i for i in range(len(parents)) if not ch[i]]
    V = 8
    for trial in range(200):
        logits = rng.standard_normal((len(parents), V))
        toks = synth.draft_tokens(parents, V, trial, "t")
        a, bonus, path = O.greedy_accept(logits, toks, parents)
        best = []
        for leaf in leaves:
            p, j = [], leaf
            while j != -1:
                p.append(j)
                j = parents[j]
            p = p[::-1]
            m = 1
            while m < len(p) and toks[p[m]] == int(np.argmax(logits[p[m - 1]])):
                m += 1
            if m > len(best):
                best = p[:m]
        assert path == best and a == len(best) - 1
        assert bonus == int(np.argmax(logits[path[-1]]))


def test_eagle_tree_shape():
    parents = synth.eagle_tree(60, (4, 3, 2, 2, 1, 1))
    assert len(parents) == 61
    O.check_parents(parents)
    d = O.depths(parents)
    assert [int((d == t).sum()) for t in range(1, 7)] == [4, 8, 9, 13, 13, 13]
    ch = O.children_of(parents)
    assert sum(1 for i in range(61) if not ch[i]) == 16


def test_inverse_cdf_never_selects_zero_mass_token():
    # u = 0 must land on the first token with positive mass, not on a leading zero-mass token
    assert O.inverse_cdf([0.0, 0.0, 0.5, 0.5], 0.0)[0] == 2
    assert O.inverse_cdf([0.25, 0.0, 0.75], 0.25)[0] == 2
    assert O.inverse_cdf([0.25, 0.0, 0.75], 0.2499)[0] == 0


def test_stored_kv_rows_are_bf16_values(tiny_oracle_weights):
    arch = synth.TINY
    kv = [O.empty_kv(arch) for _ in range(arch.n_layers)]
    _, nk = O.verify_request(tiny_oracle_weights, arch, frozenset({1}), [3, 4, 5], [-1, 0, 1], 0, kv)
    for k, v in nk.values():
        assert np.array_equal(O.round_to_bf16(k), k) and np.array_equal(O.round_to_bf16(v), v)
        assert np.any(k != 0)


def test_draw_consistency_check():
    w = np.array([0.1, 0.0, 0.4, 0.5])
    assert O.draw_consistent(w, 0.3, 2) and O.draw_consistent(w, 0.05, 0)
    assert not O.draw_consistent(w, 0.3, 3) and not O.draw_consistent(w, 0.1, 1)  # zero mass
    assert O.draw_consistent(w, 0.10005, 0, band=1e-4) and not O.draw_consistent(w, 0.2, 0, band=1e-4)
