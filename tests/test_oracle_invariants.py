"""Invariants the oracle must satisfy (no GPU): skip = deleted layers, all-skipped closed form,
tree = chain per root path, block verify = greedy autoregressive decode, KV compaction = chain of
the accepted path, and speculative sampling reproduces the target distribution."""
import dataclasses

import numpy as np
import pytest

from oracle import tss_oracle as O
from paper_2609_26100_gb300 import synth

D64 = np.float64


@pytest.fixture(scope="module")
def tiny():
    from tests.conftest import oracle_weights
    arch = synth.TINY
    return arch, oracle_weights(synth.make_weights(arch))


@pytest.fixture(scope="module")
def tiny_ctx(tiny):
    arch, w = tiny
    ctx = synth.uniform_ints(24, arch.vocab, 42, "inv.ctx").tolist()
    return ctx


def _kv(arch, w, skip, ctx):
    return O.prefill(w, arch, skip, ctx, D64)


def test_skip_equals_model_with_layers_deleted(tiny, tiny_ctx):
    arch, w = tiny
    skip = frozenset({1, 2})
    kv = _kv(arch, w, skip, tiny_ctx)
    parents = synth.chain_parents(3)
    toks = synth.draft_tokens(parents, arch.vocab, 1, "inv.del")
    got, nk = O.verify_request(w, arch, skip, toks, parents, len(tiny_ctx), kv, D64)
    keep = [0, 3]
    arch2 = dataclasses.replace(arch, n_layers=len(keep))
    w2 = dict(w, layers=[w["layers"][l] for l in keep])
    kv2 = [kv[l] for l in keep]
    ref, nk2 = O.verify_request(w2, arch2, frozenset(), toks, parents, len(tiny_ctx), kv2, D64)
    assert np.array_equal(got, ref)
    assert sorted(nk) == keep and all(np.array_equal(nk[keep[i]][0], nk2[i][0]) for i in range(2))


def test_all_layers_skipped_is_norm_of_embedding_times_lm_head(tiny):
    arch, w = tiny
    toks = [5, 17, 2047, 0]
    parents = synth.chain_parents(3)
    logits, nk = O.verify_request(w, arch, frozenset(range(arch.n_layers)), toks, parents, 0,
                                  [None] * arch.n_layers, D64)
    e = O.as_float(w["embed"], D64)[toks]
    g = O.as_float(w["final_norm"], D64)
    ref = (e / np.sqrt(np.mean(e * e, axis=1, keepdims=True) + arch.rms_eps) * g) @ O.as_float(w["lm_head"], D64).T
    assert np.allclose(logits, ref, rtol=0, atol=1e-12)
    assert nk == {}


def test_empty_mask_and_unknown_domain_are_dense(tiny, tiny_ctx):
    arch, w = tiny
    phi = {3: [0, 2]}
    kv = _kv(arch, w, frozenset(), tiny_ctx)
    parents = synth.chain_parents(2)
    toks = synth.draft_tokens(parents, arch.vocab, 2, "inv.dense")
    dense, _ = O.verify_request(w, arch, frozenset(), toks, parents, len(tiny_ctx), kv, D64)
    unk, _ = O.verify_request(w, arch, O.skip_set(phi, 9), toks, parents, len(tiny_ctx), kv, D64)
    assert np.array_equal(dense, unk)
    sk, _ = O.verify_request(w, arch, O.skip_set(phi, 3), toks, parents, len(tiny_ctx), kv, D64)
    assert not np.allclose(dense, sk)


def test_tree_logits_equal_chain_logits_of_each_root_path(tiny, tiny_ctx):
    arch, w = tiny
    skip = frozenset({2})
    kv = _kv(arch, w, skip, tiny_ctx)
    parents = synth.eagle_tree(12, (3, 2, 2))
    toks = synth.draft_tokens(parents, arch.vocab, 3, "inv.tree")
    C = len(tiny_ctx)
    tree, tree_kv = O.verify_request(w, arch, skip, toks, parents, C, kv, D64)
    for node in range(len(parents)):
        path, j = [], node
        while j != -1:
            path.append(j)
            j = parents[j]
        path = path[::-1]
        chain, chain_kv = O.verify_request(w, arch, skip, [toks[i] for i in path],
                                           synth.chain_parents(len(path) - 1), C, kv, D64)
        assert np.allclose(chain[-1], tree[node], rtol=0, atol=1e-10)
        for l in chain_kv:
            assert np.allclose(chain_kv[l][0][-1], tree_kv[l][0][node], atol=1e-10)


def _greedy_ar(arch, w, skip, kv, root, C, n):
    """Greedy autoregressive decode, one token per forward, appending each token's KV."""
    out, logits_rows, tok = [], [], root
    for s in range(n):
        lg, nk = O.verify_request(w, arch, skip, [tok], [-1], C + s, kv, D64)
        kv = O.append_kv(kv, nk, [0])
        tok = O.argmax_lowest(lg[0])
        out.append(tok)
        logits_rows.append(lg[0])
    return out, np.array(logits_rows)


@pytest.mark.parametrize("skip", [frozenset(), frozenset({2})])
def test_chain_verify_equals_greedy_autoregressive_decode(tiny, tiny_ctx, skip):
    arch, w = tiny
    kv = _kv(arch, w, skip, tiny_ctx)
    C, k = len(tiny_ctx), 4
    root = 1234
    greedy, ar_logits = _greedy_ar(arch, w, skip, kv, root, C, k + 1)
    toks = [root] + greedy[:k]
    logits, _ = O.verify_request(w, arch, skip, toks, synth.chain_parents(k), C, kv, D64)
    assert np.allclose(logits, ar_logits, rtol=0, atol=1e-10)
    a, bonus, path = O.greedy_accept(logits, toks, synth.chain_parents(k))
    assert (a, bonus, path) == (k, greedy[k], list(range(k + 1)))
    for j in range(1, k + 1):  # replace draft j: exactly j-1 drafts are accepted
        bad = list(toks)
        bad[j] = (bad[j] + 1) % arch.vocab
        lg, _ = O.verify_request(w, arch, skip, bad, synth.chain_parents(k), C, kv, D64)
        a, bonus, _ = O.greedy_accept(lg, bad, synth.chain_parents(k))
        assert a == j - 1 and bonus == greedy[j - 1]


def test_prefill_extends_consistently(tiny, tiny_ctx):
    arch, w = tiny
    skip = frozenset({0})
    block = [7, 8, 9]
    kv_full = O.prefill(w, arch, skip, tiny_ctx + block, D64)
    kv = _kv(arch, w, skip, tiny_ctx)
    _, nk = O.verify_request(w, arch, skip, block, synth.chain_parents(2), len(tiny_ctx), kv, D64)
    for l in nk:
        assert np.allclose(np.transpose(nk[l][0], (1, 0, 2)), kv_full[l][0][:, len(tiny_ctx):], atol=1e-10)
        assert np.allclose(np.transpose(nk[l][1], (1, 0, 2)), kv_full[l][1][:, len(tiny_ctx):], atol=1e-10)
    assert kv_full[0] is None


def test_tree_compaction_equals_chain_of_accepted_path(tiny, tiny_ctx):
    arch, w = tiny
    skip = frozenset({3})
    kv = _kv(arch, w, skip, tiny_ctx)
    C = len(tiny_ctx)
    parents = synth.eagle_tree(15, (3, 2, 2, 1))
    root = 77
    greedy, _ = _greedy_ar(arch, w, skip, kv, root, C, 4)
    toks = synth.draft_tokens(parents, arch.vocab, 4, "inv.compact")
    toks[0] = root
    # plant the greedy continuation along the path through child ranks (1, 0, 1, 0)
    ch = O.children_of(parents)
    cur = 0
    for rank, g in zip((1, 0, 1, 0), greedy):
        if len(ch[cur]) <= rank:
            break
        nxt = ch[cur][rank]
        for sib in ch[cur]:
            if toks[sib] == g and sib != nxt:
                toks[sib] = (g + 1) % arch.vocab
        toks[nxt] = g
        cur = nxt
    logits, nk = O.verify_request(w, arch, skip, toks, parents, C, kv, D64)
    a, bonus, path = O.greedy_accept(logits, toks, parents)
    assert a >= 2
    chain_logits, chain_kv = O.verify_request(w, arch, skip, [toks[i] for i in path],
                                              synth.chain_parents(a), C, kv, D64)
    assert np.allclose(chain_logits, logits[path], atol=1e-10)
    for l in nk:
        assert np.allclose(O.compact_block_rows(nk[l][0], path), chain_kv[l][0], atol=1e-10)
        assert np.allclose(O.compact_block_rows(nk[l][1], path), chain_kv[l][1], atol=1e-10)
    assert O.new_ctx_len(C, a) == C + 1 + a


def test_skipped_layers_produce_no_kv(tiny, tiny_ctx):
    arch, w = tiny
    skip = frozenset({1, 3})
    kv = _kv(arch, w, skip, tiny_ctx)
    assert kv[1] is None and kv[3] is None
    _, nk = O.verify_request(w, arch, skip, [1, 2], [-1, 0], len(tiny_ctx), kv, D64)
    assert sorted(nk) == [0, 2]


# ---------------------------------------------------------------------------------------------
# Speculative sampling reproduces the target distribution
# ---------------------------------------------------------------------------------------------
def _threshold(fn, lo=0.0, hi=1.0, iters=80):
    """Boundary of a monotone predicate fn (True below, False above) on [lo, hi)."""
    if not fn(lo):
        return lo
    if fn(np.nextafter(hi, 0)):
        return hi
    for _ in range(iters):
        mid = 0.5 * (lo + hi)
        if fn(mid):
            lo = mid
        else:
            hi = mid
    return 0.5 * (lo + hi)


def _first_emitted_distribution(logits, q, V):
    """Exact distribution of the first token emitted by spec_sample_accept (k = 1), measured by
    locating the oracle's decision boundaries in r and u by bisection."""
    dist = np.zeros(V)
    for x in range(V):
        toks = [0, x]
        base = np.full(3, 0.5)

        def accepts(r):
            u = base.copy()
            u[0] = r
            return O.spec_sample_accept(logits, toks, q, u)[0] == 1

        acc = _threshold(accepts)
        dist[x] += q[1][x] * acc
        if acc < 1.0:
            rej = np.array([np.nextafter(1.0, 0), 0.5, 0.5])
            prev = 0.0
            for v in range(V):
                def below(uu, v=v):
                    u = rej.copy()
                    u[1] = uu
                    return O.spec_sample_accept(logits, toks, q, u)[1] <= v
                b = _threshold(below)
                dist[v] += q[1][x] * (1 - acc) * (b - prev)
                prev = b
    return dist


@pytest.mark.parametrize("V", [3, 4, 6])
def test_spec_sampling_first_token_is_target_distributed(V):
    rng = np.random.default_rng(V)
    for _ in range(3):
        logits = rng.standard_normal((2, V)) * 2
        q = np.zeros((2, V))
        q[1] = rng.dirichlet(np.ones(V))
        p = O.softmax_t(logits[0], 1.0)
        assert np.allclose(_first_emitted_distribution(logits, q, V), p, atol=1e-12)


def test_spec_sampling_second_token_given_first_accepted():
    V = 4
    rng = np.random.default_rng(11)
    logits = rng.standard_normal((3, V))
    q = np.zeros((3, V))
    q[1], q[2] = rng.dirichlet(np.ones(V)), rng.dirichlet(np.ones(V))
    p1 = O.softmax_t(logits[1], 1.0)
    dist = np.zeros(V)
    x1 = 2
    for x in range(V):
        toks = [0, x1, x]

        def accepts(r):
            u = np.full(5, 0.5)
            u[0], u[1] = 0.0, r
            return O.spec_sample_accept(logits, toks, q, u)[0] == 2

        acc = _threshold(accepts)
        dist[x] += q[2][x] * acc
        prev = 0.0
        for v in range(V):
            def below(uu, v=v):
                u = np.full(5, 0.5)
                u[0], u[1], u[3] = 0.0, np.nextafter(1.0, 0), uu
                return O.spec_sample_accept(logits, toks, q, u)[1] <= v
            b = _threshold(below)
            dist[v] += q[2][x] * (1 - acc) * (b - prev)
            prev = b
    assert np.allclose(dist, p1, atol=1e-12)


def test_spec_sampling_all_accepted_bonus_from_last_row():
    V = 5
    logits = np.log(np.array([[0.1, 0.2, 0.3, 0.2, 0.2], [0.5, 0.1, 0.1, 0.1, 0.2]]))
    q = np.zeros((2, V))
    q[1] = np.array([0.05, 0.05, 0.05, 0.8, 0.05])
    u = np.array([0.0, 0.5, 0.55])  # accept (r = 0); bonus ~ p_1 at u = 0.55 -> token 1
    a, bonus, path, _ = O.spec_sample_accept(logits, [0, 2], q, u)
    assert (a, bonus, path) == (1, 1, [0, 1])


def test_spec_sampling_monte_carlo_with_philox():
    V, k, T = 4, 2, 1.0
    rng = np.random.default_rng(12)
    logits = rng.standard_normal((k + 1, V))
    q = np.zeros((k + 1, V))
    q[1:] = rng.dirichlet(np.ones(V), size=k)
    p0 = O.softmax_t(logits[0], T)
    n = 20000
    counts = np.zeros(V)
    draws = np.random.default_rng(13)
    for step in range(n):
        x1 = int(draws.choice(V, p=q[1]))
        x2 = int(draws.choice(V, p=q[2]))
        u = O.philox_uniforms(seed=7, offset=step, req=0, k=k)
        a, bonus, _, _ = O.spec_sample_accept(logits, [0, x1, x2], q, u, T)
        counts[x1 if a >= 1 else bonus] += 1
    chi2 = float(np.sum((counts - n * p0) ** 2 / (n * p0)))
    from scipy.stats import chi2 as chi2d
    assert chi2d.sf(chi2, V - 1) > 1e-3


def test_layer_major_batch_equals_per_request_verification(tiny, tiny_ctx):
    """verify_requests (layer by layer over a batch) gives each request exactly what
    verify_request gives it alone: mixed skip sets (one dense, one skipping every layer), context
    lengths and a tree block."""
    arch, w = tiny
    skips = [frozenset({1}), frozenset(), frozenset({0, 3}), frozenset(range(arch.n_layers))]
    blocks, kvs = [], []
    for b, skip in enumerate(skips):
        ctx = tiny_ctx[: 24 - 5 * b]
        parents = synth.eagle_tree(9, (3, 2, 1)) if b == 2 else synth.chain_parents(3 + b)
        toks = synth.draft_tokens(parents, arch.vocab, 5, f"inv.batch{b}")
        blocks.append((toks, parents, len(ctx)))
        kvs.append(_kv(arch, w, skip, ctx))
    got = O.verify_requests(w, arch, skips, blocks, lambda b, l: kvs[b][l], D64)
    for b, skip in enumerate(skips):
        toks, parents, C = blocks[b]
        ref, nk = O.verify_request(w, arch, skip, toks, parents, C, kvs[b], D64)
        assert np.array_equal(got[b][0], ref)
        assert sorted(got[b][1]) == sorted(nk)
        for l in nk:
            assert np.array_equal(got[b][1][l][0], nk[l][0]) and np.array_equal(got[b][1][l][1], nk[l][1])
