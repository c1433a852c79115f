"""Planted mistakes in the oracle (CPU only): each case replaces one oracle function with a
plausible wrong variant -- a dropped term, a wrong sign, index or operand, an off-by-one -- and
checks that at least one of the pins in test_oracle_pins.py / test_oracle_invariants.py then
fails.  This is a test of the pins: an oracle mistake of any of these kinds cannot pass them."""
import math

import numpy as np
import pytest

from oracle import philox
from oracle import tss_oracle as O
from paper_2609_26100_gb300 import synth
from tests import test_oracle_invariants as I
from tests import test_oracle_pins as P

_ORIG = {name: getattr(O, name) for name in ("verify_request", "apply_rope", "block_attention")}


@pytest.fixture(scope="module")
def tiny_setup():
    from tests.conftest import oracle_weights
    arch = synth.TINY
    w = oracle_weights(synth.make_weights(arch))
    ctx = synth.uniform_ints(24, arch.vocab, 42, "inv.ctx").tolist()
    return (arch, w), ctx, w


# ------------------------------------------------------------------------------------------------
# Mutants (each wrong in exactly one way)
# ------------------------------------------------------------------------------------------------
def rms_no_gain(h, g, eps):
    return h / np.sqrt(np.mean(h * h, axis=-1, keepdims=True) + eps)


def rms_eps_outside_root(h, g, eps):
    return h / (np.sqrt(np.mean(h * h, axis=-1, keepdims=True)) + eps) * g


def rms_sum_not_mean(h, g, eps):
    return h / np.sqrt(np.sum(h * h, axis=-1, keepdims=True) + eps) * g


def rope_interleaved_pairs(x, cos, sin):
    xe, xo = x[..., 0::2], x[..., 1::2]
    c, s = cos[:, None, :], sin[:, None, :]
    out = np.empty_like(x)
    out[..., 0::2] = xe * c - xo * s
    out[..., 1::2] = xo * c + xe * s
    return out


def rope_reverse_rotation(x, cos, sin):
    return _ORIG["apply_rope"](x, cos, -sin)


def rope_freq_without_factor_two(positions, head_dim, theta, dt=np.float32):
    half = head_dim // 2
    inv_freq = float(theta) ** (-np.arange(half, dtype=np.float64) / head_dim)
    ang = np.asarray(positions, dtype=np.float64)[:, None] * inv_freq[None, :]
    return np.cos(ang).astype(dt), np.sin(ang).astype(dt)


def attention_unscaled(q, k_ctx, v_ctx, k_blk, v_blk, allowed):
    D = q.shape[-1]
    return _ORIG["block_attention"](q * math.sqrt(D), k_ctx, v_ctx, k_blk, v_blk, allowed)


def attention_causal_by_index(q, k_ctx, v_ctx, k_blk, v_blk, allowed):
    N = q.shape[0]
    return _ORIG["block_attention"](q, k_ctx, v_ctx, k_blk, v_blk, np.tril(np.ones((N, N), dtype=bool)))


def attention_without_self(q, k_ctx, v_ctx, k_blk, v_blk, allowed):
    a = np.array(allowed, dtype=bool)
    if k_ctx.shape[1] == 0:  # nothing else to attend to: keep the row well defined
        return np.zeros_like(q)
    np.fill_diagonal(a, False)
    return _ORIG["block_attention"](q, k_ctx, v_ctx, k_blk, v_blk, a)


def silu_as_sigmoid(x):
    return 1.0 / (1.0 + np.exp(-x))


def round_bf16_truncate(x):
    x = np.ascontiguousarray(x, dtype=np.float32)
    return (x.view(np.uint32) & np.uint32(0xFFFF0000)).view(np.float32)


def verify_ignores_skip(weights, arch, skip, *args, **kw):
    return _ORIG["verify_request"](weights, arch, frozenset(), *args, **kw)


def verify_skips_one_too_many(weights, arch, skip, *args, **kw):
    extra = frozenset({max(skip) + 1}) if skip and max(skip) + 1 < arch.n_layers else frozenset()
    return _ORIG["verify_request"](weights, arch, frozenset(skip) | extra, *args, **kw)


def argmax_highest_on_ties(row):
    r = np.asarray(row)
    return int(len(r) - 1 - np.argmax(r[::-1]))


def greedy_own_row(logits, tokens, parents):
    ch = O.children_of(parents)
    cur, path = 0, [0]
    while True:
        nxt = next((c for c in ch[cur] if int(tokens[c]) == O.argmax_lowest(logits[c])), None)
        if nxt is None:
            return len(path) - 1, O.argmax_lowest(logits[cur]), path
        cur = nxt
        path.append(cur)


def greedy_first_child_only(logits, tokens, parents):
    ch = O.children_of(parents)
    cur, path = 0, [0]
    while ch[cur] and int(tokens[ch[cur][0]]) == O.argmax_lowest(logits[cur]):
        cur = ch[cur][0]
        path.append(cur)
    return len(path) - 1, O.argmax_lowest(logits[cur]), path


def _spec_sample(logits, tokens, q, uniforms, temperature=1.0, return_draw=False, *, accept, residual, bonus_row):
    """Speculative sampling with pluggable accept test, residual and bonus row (for mutants)."""
    k = len(tokens) - 1
    for i in range(1, k + 1):
        p = O.softmax_t(logits[i - 1], temperature)
        x = int(tokens[i])
        if accept(float(uniforms[i - 1]), float(q[i][x]), float(p[x])):
            continue
        res = residual(p, np.asarray(q[i], dtype=np.float64))
        v = O.inverse_cdf(res, float(uniforms[k + i - 1]))[0]
        return i - 1, v, list(range(i)), False
    p = O.softmax_t(logits[bonus_row(k)], temperature)
    v = O.inverse_cdf(p, float(uniforms[2 * k]))[0]
    return k, v, list(range(k + 1)), False


def spec_inverted_ratio(*a, **kw):
    return _spec_sample(*a, **kw, accept=lambda r, qx, px: r * px < qx,
                        residual=lambda p, q: np.maximum(p - q, 0.0), bonus_row=lambda k: k)


def spec_residual_not_clipped(*a, **kw):
    return _spec_sample(*a, **kw, accept=lambda r, qx, px: r * qx < px,
                        residual=lambda p, q: np.abs(p - q), bonus_row=lambda k: k)


def spec_residual_is_target(*a, **kw):
    return _spec_sample(*a, **kw, accept=lambda r, qx, px: r * qx < px,
                        residual=lambda p, q: p, bonus_row=lambda k: k)


def spec_bonus_from_previous_row(*a, **kw):
    return _spec_sample(*a, **kw, accept=lambda r, qx, px: r * qx < px,
                        residual=lambda p, q: np.maximum(p - q, 0.0), bonus_row=lambda k: k - 1)


def inverse_cdf_left(weights, u):
    c = np.cumsum(np.asarray(weights, dtype=np.float64))
    v = min(int(np.searchsorted(c, u * c[-1], side="left")), len(c) - 1)
    lo = c[v - 1] if v > 0 else 0.0
    return v, u, lo / c[-1], c[v] / c[-1]


def compact_identity(rows, path):
    return np.asarray(rows)[: len(path)]


def ctx_len_without_root(ctx_len, accept_len):
    return ctx_len + accept_len


def sparsity_over_active(skip, n_layers):
    return len(set(skip)) / float(n_layers - len(set(skip)))


def union_as_intersection(skips, n_layers):
    return [l for l in range(n_layers) if all(l not in s for s in skips)]


def unknown_domain_skips_all(phi, domain):
    return frozenset(int(l) for l in phi[domain]) if domain in phi else frozenset(range(64))


def ancestors_without_self(parents):
    a = np.array(_ORIG_ANC(parents), dtype=bool)
    np.fill_diagonal(a, False)
    return a


_ORIG_ANC = O.ancestor_or_self


# ------------------------------------------------------------------------------------------------
# Cases: (patches [(module, name, mutant)], pins that must catch it)
# ------------------------------------------------------------------------------------------------
def _pins_block(t):
    (tiny, ctx, w) = t
    return [P.test_single_token_block_closed_form,
            lambda: I.test_skip_equals_model_with_layers_deleted(tiny, ctx)]


CASES = {
    "rmsnorm drops the gain": ([(O, "rms_norm", rms_no_gain)], lambda t: [P.test_rmsnorm_closed_forms]),
    "rmsnorm eps outside the root": ([(O, "rms_norm", rms_eps_outside_root)], lambda t: [P.test_rmsnorm_closed_forms]),
    "rmsnorm sum instead of mean": ([(O, "rms_norm", rms_sum_not_mean)], lambda t: [P.test_rmsnorm_closed_forms]),
    "rope pairs adjacent elements": ([(O, "apply_rope", rope_interleaved_pairs)],
                                     lambda t: [P.test_rope_is_complex_rotation_of_half_pairs]),
    "rope rotates the wrong way": ([(O, "apply_rope", rope_reverse_rotation)],
                                   lambda t: [P.test_rope_is_complex_rotation_of_half_pairs]),
    "rope frequency exponent -i/D": ([(O, "rope_cos_sin", rope_freq_without_factor_two)],
                                     lambda t: [P.test_rope_is_complex_rotation_of_half_pairs]),
    "attention without 1/sqrt(D)": ([(O, "block_attention", attention_unscaled)],
                                    lambda t: [lambda: P.test_block_attention_matches_brute_force([-1, 0, 1, 2])]),
    "tree mask replaced by a causal mask": ([(O, "block_attention", attention_causal_by_index)],
                                            lambda t: [lambda: P.test_block_attention_matches_brute_force([-1, 0, 0, 1, 1, 2, 5])]),
    "attention excludes the row itself": ([(O, "block_attention", attention_without_self)],
                                          lambda t: [P.test_attention_without_context_returns_own_value,
                                                     lambda: P.test_block_attention_matches_brute_force([-1, 0, 1, 2])]),
    "ancestor mask without self": ([(O, "ancestor_or_self", ancestors_without_self)],
                                   lambda t: [lambda: P.test_block_attention_matches_brute_force([-1, 0, 1, 2])]),
    "silu is the sigmoid": ([(O, "silu", silu_as_sigmoid)], lambda t: [P.test_silu_closed_forms]),
    "bf16 rounding truncates": ([(O, "round_to_bf16", round_bf16_truncate)],
                                lambda t: [P.test_round_to_bf16_ties_and_library_agreement]),
    "skip set ignored": ([(O, "verify_request", verify_ignores_skip)], _pins_block),
    "one layer too many skipped": ([(O, "verify_request", verify_skips_one_too_many)],
                                   lambda t: [lambda: I.test_skip_equals_model_with_layers_deleted(t[0], t[1])]),
    "argmax ties to the highest id": ([(O, "argmax_lowest", argmax_highest_on_ties)],
                                      lambda t: [P.test_argmax_ties_and_margin]),
    "greedy walk reads the child's own row": ([(O, "greedy_accept", greedy_own_row)],
                                              lambda t: [P.test_tree_accept_equals_longest_matching_root_path]),
    "greedy walk tries the first child only": ([(O, "greedy_accept", greedy_first_child_only)],
                                               lambda t: [P.test_tree_accept_equals_longest_matching_root_path]),
    "sampling accept ratio inverted": ([(O, "spec_sample_accept", spec_inverted_ratio)],
                                       lambda t: [lambda: I.test_spec_sampling_first_token_is_target_distributed(4)]),
    "sampling residual not clipped at zero": ([(O, "spec_sample_accept", spec_residual_not_clipped)],
                                              lambda t: [lambda: I.test_spec_sampling_first_token_is_target_distributed(4)]),
    "sampling residual is the target": ([(O, "spec_sample_accept", spec_residual_is_target)],
                                        lambda t: [lambda: I.test_spec_sampling_first_token_is_target_distributed(4)]),
    "sampling bonus from the previous row": ([(O, "spec_sample_accept", spec_bonus_from_previous_row)],
                                             lambda t: [I.test_spec_sampling_all_accepted_bonus_from_last_row]),
    "inverse CDF lands on a zero-mass token": ([(O, "inverse_cdf", inverse_cdf_left)],
                                               lambda t: [P.test_inverse_cdf_never_selects_zero_mass_token]),
    "KV compaction keeps block order": ([(O, "compact_block_rows", compact_identity)],
                                        lambda t: [lambda: I.test_tree_compaction_equals_chain_of_accepted_path(t[0], t[1])]),
    "committed length forgets the root": ([(O, "new_ctx_len", ctx_len_without_root)],
                                          lambda t: [lambda: I.test_tree_compaction_equals_chain_of_accepted_path(t[0], t[1])]),
    "sparsity ratio over active layers": ([(O, "sparsity_ratio", sparsity_over_active)],
                                          lambda t: [P.test_sparsity_ratio_reproduces_table1]),
    "batch union taken as an intersection": ([(O, "union_active_layers", union_as_intersection)],
                                             lambda t: [P.test_union_and_row_lists_brute_force]),
    "unknown domain skips every layer": ([(O, "skip_set", unknown_domain_skips_all)],
                                         lambda t: [P.test_unknown_domain_falls_back_to_dense]),
    "philox multiplier M0 wrong": ([(philox, "M0", 0xD2511F55)], lambda t: [P.test_philox_known_answers]),
    "philox Weyl constant W1 wrong": ([(philox, "W1", 0xBB67AE87)], lambda t: [P.test_philox_known_answers]),
}


def _fails(fn):
    try:
        fn()
    except Exception:  # an assertion or any error the mistake causes
        return True
    return False


@pytest.mark.parametrize("case", sorted(CASES))
def test_planted_mistake_is_caught(case, tiny_setup, monkeypatch):
    patches, pins = CASES[case]
    checks = pins(tiny_setup)
    # the unmutated oracle passes these pins
    assert not any(_fails(fn) for fn in checks), "pin fails without the mutation"
    for mod, name, mutant in patches:
        monkeypatch.setattr(mod, name, mutant)
    assert any(_fails(fn) for fn in checks), f"no pin catches: {case}"
