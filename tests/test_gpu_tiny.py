"""GPU parity on the tiny decoder (4 layers, d 256, 4 heads x 64, MLP 688, vocab 2048): the CUDA
path through the C ABI against the CPU oracle on the same seeded inputs."""
import os

import numpy as np
import pytest
import torch

from oracle import tss_oracle as O
from paper_2609_26100_gb300 import native, synth
from tests.conftest import oracle_weights
from tests.parity_util import assert_logits, check_sample, greedy_valid, gpu_path, kv_to_torch, to_device_weights

pytestmark = pytest.mark.gpu

ARCH = synth.TINY
SEED = synth.DEFAULT_SEED


@pytest.fixture(scope="module")
def weights():
    from paper_2609_26100_gb300 import build
    build.build()
    w = synth.make_weights(ARCH)
    return w, oracle_weights(w), to_device_weights(w)


PATHS = ["persistent", "hybrid", "multi"]


def make_runner(wg, n_slots=4, cap=512, path="persistent", **kw):
    """path: "persistent" (one cooperative kernel for all layers), "hybrid" (persistent-kernel
    launches over the GEMM phases with each layer's attention as its own kernel, the long-context
    plan) or "multi" (kernel per op)."""
    from paper_2609_26100_gb300.runner import TssRunner
    os.environ["TSS_PATH"] = "persistent" if path == "hybrid" else path
    os.environ["TSS_ATTN"] = "external" if path == "hybrid" else "internal"
    try:
        return TssRunner(ARCH, wg, n_slots=n_slots, kv_cap=cap, max_batch=8, **kw)
    finally:
        os.environ.pop("TSS_PATH", None)
        os.environ.pop("TSS_ATTN", None)


def upload_context(run, kv, slot):
    for l, layer in enumerate(kv):
        if layer is not None:
            k, v = kv_to_torch(layer)
            run.write_kv(l, slot, k, v)


def greedy_ar(wo, skip, kv, root, C, n):
    out, tok = [], root
    for s in range(n):
        lg, nk = O.verify_request(wo, ARCH, skip, [tok], [-1], C + s, kv)
        kv = O.append_kv(kv, nk, [0])
        tok = O.argmax_lowest(lg[0])
        out.append(tok)
    return out


def run_step(run, reqs, **kw):
    depth = max(max(synth.depths_of(r.parents)) for r in reqs)
    res = run.alloc_results(len(reqs), sum(len(r.parents) for r in reqs), path_stride=max(64, depth + 1))
    b = run.batch(reqs, **kw)
    run.verify(b, res)
    st = run.sync_status()
    torch.cuda.synchronize()
    return res, st


@pytest.mark.parametrize("path", PATHS)
@pytest.mark.parametrize("mask_layers", [(2,), ()])
def test_chain_greedy_16_steps_lockstep(weights, mask_layers, path):
    """Tiny config: 128-token context (oracle prefill under the mask), chain k=4 = oracle greedy
    continuation with the token at a seeded position replaced, 16 verify steps."""
    w, wo, wg = weights
    wl = synth.workload_tiny(mask_layers)
    skip = O.mask_to_set(wl.phi[0])
    ctx = synth.uniform_ints(128, ARCH.vocab, SEED, "tiny.ctx").tolist()
    kv = O.prefill(wo, ARCH, skip, ctx)
    run = make_runner(wg, n_slots=1, cap=256, path=path)
    run.set_phi(wl.phi)
    upload_context(run, kv, 0)
    C, k = len(ctx), 4
    root = int(synth.uniform_ints(1, ARCH.vocab, SEED, "tiny.root").item())
    flagged = exact = 0
    pos_draws = synth.uniform_ints(16, k, SEED, "tiny.pos").tolist()
    for step in range(16):
        greedy = greedy_ar(wo, skip, kv, root, C, k)
        j = 1 + pos_draws[step]
        toks = [root] + greedy
        toks[j] = (toks[j] + 1 + step) % ARCH.vocab
        parents = synth.chain_parents(k)
        ref, nk = O.verify_request(wo, ARCH, skip, toks, parents, C, kv)
        a, bonus, path = O.greedy_accept(ref, toks, parents)
        assert a == j - 1  # the replaced draft is the first mismatch
        res, st = run_step(run, [synth.Request(C, parents, toks, 0)])
        assert st == native.TSS_OK
        gl = res["logits"].cpu().numpy()
        assert_logits(gl, ref, f"step {step}")
        ga, gb = int(res["accept_len"][0]), int(res["bonus"][0])
        gp = gpu_path(res, 0, ga)
        if O.greedy_flagged(ref, path):
            flagged += 1
            assert greedy_valid(ref, toks, parents, gp, gb)
        else:
            exact += 1
            assert (ga, gb, gp) == (a, bonus, path)
        assert int(res["new_ctx_len"][0]) == C + 1 + ga
        # KV rows the GPU appended for the block, every layer the request runs
        for l in nk:
            gk = run.kv[l][0, 0, :, C:C + k + 1].float().cpu().numpy()
            np.testing.assert_allclose(gk, np.transpose(nk[l][0], (1, 0, 2)), atol=3e-2, rtol=2e-2)
        for l in skip:
            assert torch.count_nonzero(run.kv[l]) == 0  # a skipped layer's cache is never written
        # lockstep on the oracle's state
        kv = O.append_kv(kv, nk, path)
        for l in nk:
            kk, vv = kv_to_torch((np.transpose(nk[l][0][path], (1, 0, 2)), np.transpose(nk[l][1][path], (1, 0, 2))))
            run.write_kv(l, 0, kk, vv, pos0=C)
        C += 1 + a
        root = bonus
    print(f"[parity] tiny chain {mask_layers}: {exact} exact, {flagged} flagged (top-2 margin < {O.GREEDY_MARGIN})")
    assert exact + flagged == 16 and exact >= 12
    run.close()


def test_greedy_exact_over_many_blocks(weights):
    """48 request-steps (8 requests of two domains and the dense path, contexts 3-200, chains of
    1-6 drafts, half of them starting with a greedy prefix of seeded length): accept_len, bonus
    and path equal the oracle's on every step whose walk reads no near-tie row (top-2 margin <
    0.05, flagged, counted, and checked for validity instead)."""
    w, wo, wg = weights
    phi = {0: O.set_to_mask({2}), 1: O.set_to_mask({0, 3})}
    doms = [0, 1, 5, 0, 1, 5, 0, 1]
    ctxs = [200, 3, 64, 131, 17, 90, 45, 8]
    run = make_runner(wg, n_slots=8, cap=256)
    run.set_phi(phi)
    skips, kvs = [], []
    for b in range(8):
        skip = O.skip_set({d: O.mask_to_set(m) for d, m in phi.items()}, doms[b])
        kv = O.prefill(wo, ARCH, skip, synth.uniform_ints(ctxs[b], ARCH.vocab, SEED, f"many.ctx{b}").tolist())
        upload_context(run, kv, b)
        skips.append(skip)
        kvs.append(kv)
    exact = flagged = 0
    for step in range(6):
        reqs = []
        for b in range(8):
            k = 1 + (b + step) % 6
            parents = synth.chain_parents(k)
            toks = synth.draft_tokens(parents, ARCH.vocab, SEED, f"many.tok{step}.{b}")
            if (b + step) % 2 == 0:
                lp = 1 + int(synth.uniform_ints(1, k, SEED, f"many.lp{step}.{b}").item())
                toks[1:1 + lp] = greedy_ar(wo, skips[b], kvs[b], toks[0], ctxs[b], lp)
            reqs.append(synth.Request(ctxs[b], parents, toks, doms[b]))
        res, st = run_step(run, reqs)
        assert st == native.TSS_OK
        gl = res["logits"].cpu().numpy()
        off = 0
        for b, r in enumerate(reqs):
            n = len(r.parents)
            ref, _ = O.verify_request(wo, ARCH, skips[b], r.tokens, r.parents, r.ctx_len, kvs[b])
            assert_logits(gl[off:off + n], ref, f"step {step} request {b}")
            a, bonus, pth = O.greedy_accept(ref, r.tokens, r.parents)
            ga, gb = int(res["accept_len"][b]), int(res["bonus"][b])
            gp = gpu_path(res, b, ga)
            if O.greedy_flagged(ref, pth):
                flagged += 1
                assert greedy_valid(ref, r.tokens, r.parents, gp, gb)
            else:
                exact += 1
                assert (ga, gb, gp) == (a, bonus, pth), f"step {step} request {b}"
            off += n
    print(f"[parity] greedy over 48 request-steps: {exact} exact, {flagged} flagged")
    assert exact + flagged == 48 and exact >= 16
    run.close()


@pytest.mark.parametrize("path", PATHS)
def test_tree_greedy_and_compaction(weights, path):
    """60-node draft tree (branching 4,3,2,2,1,1) with a planted greedy path: per-node logits,
    longest matching root path, and the KV compacted to that path."""
    w, wo, wg = weights
    skip = frozenset({1})
    ctx = synth.uniform_ints(96, ARCH.vocab, SEED, "tree.ctx").tolist()
    kv = O.prefill(wo, ARCH, skip, ctx)
    run = make_runner(wg, n_slots=2, cap=256, path=path)
    run.set_phi({3: O.set_to_mask(skip)})
    upload_context(run, kv, 1)
    parents = synth.eagle_tree(60, (4, 3, 2, 2, 1, 1))
    C = len(ctx)
    root = 11
    greedy = greedy_ar(wo, skip, kv, root, C, 6)
    toks = synth.draft_tokens(parents, ARCH.vocab, SEED, "tree.tok")
    toks[0] = root
    ch = O.children_of(parents)
    cur = 0
    for rank, g in zip((2, 1, 0, 1, 0, 0), greedy):
        if len(ch[cur]) <= rank:
            break
        nxt = ch[cur][rank]
        for sib in ch[cur]:
            if toks[sib] == g:
                toks[sib] = (g + 7) % ARCH.vocab
        toks[nxt] = g
        cur = nxt
    ref, nk = O.verify_request(wo, ARCH, skip, toks, parents, C, kv)
    a, bonus, path = O.greedy_accept(ref, toks, parents)
    res, st = run_step(run, [synth.Request(C, parents, toks, 3)], slots=[1])
    assert st == native.TSS_OK
    assert_logits(res["logits"].cpu().numpy(), ref, "tree")
    ga, gb = int(res["accept_len"][0]), int(res["bonus"][0])
    gp = gpu_path(res, 0, ga)
    if O.greedy_flagged(ref, path):
        assert greedy_valid(ref, toks, parents, gp, gb)
    else:
        assert (ga, gb, gp) == (a, bonus, path)
        assert a >= 2
    for l in nk:
        comp_k = O.compact_block_rows(nk[l][0], gp)  # oracle rows in the GPU's accepted order
        comp_v = O.compact_block_rows(nk[l][1], gp)
        gk = run.kv[l][1, 0, :, C:C + ga + 1].float().cpu().numpy()
        gv = run.kv[l][1, 1, :, C:C + ga + 1].float().cpu().numpy()
        np.testing.assert_allclose(gk, np.transpose(comp_k, (1, 0, 2)), atol=3e-2, rtol=2e-2)
        np.testing.assert_allclose(gv, np.transpose(comp_v, (1, 0, 2)), atol=3e-2, rtol=2e-2)
    assert torch.count_nonzero(run.kv[1][1]) == 0 and torch.count_nonzero(run.kv[0][0]) == 0
    run.close()


@pytest.mark.parametrize("path", PATHS)
def test_mixed_domain_batch_and_untouched_skipped_kv(weights, path):
    """Four requests with different skip sets (one domain never configured = dense), different
    context lengths and draft lengths in one batch; skipped layers' KV keeps a sentinel."""
    w, wo, wg = weights
    phi = {0: O.set_to_mask({2}), 1: O.set_to_mask({0, 3}), 2: 0}
    doms = [0, 1, 2, 7]
    ctxs = [128, 77, 200, 5]
    ks = [4, 2, 0, 3]
    run = make_runner(wg, n_slots=4, cap=256, path=path)
    run.set_phi(phi)
    sentinel = 7.0
    for t in run.kv:
        t.fill_(sentinel)
    reqs, kvs, skips = [], [], []
    for b in range(4):
        skip = O.skip_set({d: O.mask_to_set(m) for d, m in phi.items()}, doms[b])
        ctx = synth.uniform_ints(ctxs[b], ARCH.vocab, SEED, f"mix.ctx{b}").tolist()
        kv = O.prefill(wo, ARCH, skip, ctx)
        upload_context(run, kv, b)
        parents = synth.chain_parents(ks[b])
        toks = synth.draft_tokens(parents, ARCH.vocab, SEED, f"mix.tok{b}")
        reqs.append(synth.Request(ctxs[b], parents, toks, doms[b]))
        kvs.append(kv)
        skips.append(skip)
    res, st = run_step(run, reqs)
    assert st == native.TSS_OK
    gl = res["logits"].cpu().numpy()
    off = 0
    for b, r in enumerate(reqs):
        n = len(r.parents)
        ref, nk = O.verify_request(wo, ARCH, skips[b], r.tokens, r.parents, r.ctx_len, kvs[b])
        assert_logits(gl[off:off + n], ref, f"request {b}")
        a, bonus, path = O.greedy_accept(ref, r.tokens, r.parents)
        if not O.greedy_flagged(ref, path):
            assert (int(res["accept_len"][b]), int(res["bonus"][b])) == (a, bonus)
        for l in range(ARCH.n_layers):
            region = run.kv[l][b]
            if l in skips[b]:
                assert bool((region == sentinel).all()), f"request {b} skipped layer {l} was touched"
            else:
                assert bool((region[:, :, r.ctx_len + n:] == sentinel).all())
        off += n
    run.close()


@pytest.mark.parametrize("path", PATHS)
def test_maximum_block_rows(weights, path):
    """Blocks at the size limits: a 64-node chain (the most nodes a request may have), a 63-node
    draft tree and a 64-node chain of a second domain in one batch -- 192 rows, so the
    activations take the two-block hi/lo layout and every fix-up runs twelve 16-row chunks."""
    w, wo, wg = weights
    phi = {0: O.set_to_mask({1}), 1: O.set_to_mask({0, 2})}
    doms = [0, 1, 0]
    ctxs = [40, 9, 0]
    shapes = [synth.chain_parents(63), synth.eagle_tree(62, (4, 3, 2, 2, 1, 1)), synth.chain_parents(63)]
    run = make_runner(wg, n_slots=3, cap=160, path=path, max_nodes=64)
    run.set_phi(phi)
    reqs, kvs, skips = [], [], []
    for b in range(3):
        skip = O.skip_set({d: O.mask_to_set(m) for d, m in phi.items()}, doms[b])
        if ctxs[b]:
            kv = O.prefill(wo, ARCH, skip, synth.uniform_ints(ctxs[b], ARCH.vocab, SEED, f"max.ctx{b}").tolist())
            upload_context(run, kv, b)
        else:
            kv = [O.empty_kv(ARCH) for _ in range(ARCH.n_layers)]
        parents = shapes[b]
        toks = synth.draft_tokens(parents, ARCH.vocab, SEED, f"max.tok{b}")
        reqs.append(synth.Request(ctxs[b], parents, toks, doms[b]))
        kvs.append(kv)
        skips.append(skip)
    res, st = run_step(run, reqs)
    assert st == native.TSS_OK
    gl = res["logits"].cpu().numpy()
    off = 0
    for b, r in enumerate(reqs):
        n = len(r.parents)
        ref, nk = O.verify_request(wo, ARCH, skips[b], r.tokens, r.parents, r.ctx_len, kvs[b])
        assert_logits(gl[off:off + n], ref, f"request {b} ({n} nodes)")
        a, bonus, pth = O.greedy_accept(ref, r.tokens, r.parents)
        if O.greedy_flagged(ref, pth):
            ga = int(res["accept_len"][b])
            assert greedy_valid(ref, r.tokens, r.parents, gpu_path(res, b, ga), int(res["bonus"][b]))
        else:
            assert (int(res["accept_len"][b]), int(res["bonus"][b])) == (a, bonus)
        assert int(res["new_ctx_len"][b]) == r.ctx_len + 1 + int(res["accept_len"][b])
        off += n
    run.close()


@pytest.mark.parametrize("path", PATHS)
def test_gpu_prefill_matches_oracle_prefill(weights, path):
    """tss_prefill under each request's skip set: a 150-token prompt on an empty cache, 40 tokens
    appended to a 20-token context of another domain, and an empty prompt.  The K/V rows match
    the oracle's prefill, skipped layers stay untouched, and a verification step on top of the
    GPU-filled cache gives the oracle's logits."""
    w, wo, wg = weights
    phi = {0: O.set_to_mask({2}), 1: O.set_to_mask({0, 3})}
    run = make_runner(wg, n_slots=3, cap=256, path=path)
    run.set_phi(phi)
    sentinel = 7.0
    for t in run.kv:
        t.fill_(sentinel)
    doms = [0, 1, 0]
    full = [synth.uniform_ints(150, ARCH.vocab, SEED, "pf.a").tolist(),
            synth.uniform_ints(60, ARCH.vocab, SEED, "pf.b").tolist(),
            synth.uniform_ints(12, ARCH.vocab, SEED, "pf.c").tolist()]
    have = [0, 20, 12]  # tokens already in the cache (uploaded from the oracle)
    skips = [O.skip_set({d: O.mask_to_set(m) for d, m in phi.items()}, d) for d in doms]
    for b in (1, 2):
        upload_context(run, O.prefill(wo, ARCH, skips[b], full[b][:have[b]]), b)
    run.prefill([full[b][have[b]:] for b in range(3)], have, doms)
    assert run.sync_status() == native.TSS_OK
    torch.cuda.synchronize()
    for b in range(3):
        ref = O.prefill(wo, ARCH, skips[b], full[b])
        C = len(full[b])
        for l in range(ARCH.n_layers):
            region = run.kv[l][b]
            if l in skips[b]:
                assert bool((region == sentinel).all()), f"request {b} skipped layer {l} was touched"
                continue
            gk = region[0, :, :C].float().cpu().numpy()
            gv = region[1, :, :C].float().cpu().numpy()
            np.testing.assert_allclose(gk, ref[l][0], atol=5e-2, rtol=3e-2)
            np.testing.assert_allclose(gv, ref[l][1], atol=5e-2, rtol=3e-2)
            assert float(np.abs(gk - ref[l][0]).mean()) < 2e-3
            assert bool((region[:, :, C:] == sentinel).all())
    # a verification step on the GPU-filled cache of request 0
    C = len(full[0])
    parents = synth.chain_parents(4)
    toks = synth.draft_tokens(parents, ARCH.vocab, SEED, "pf.tok")
    res, st = run_step(run, [synth.Request(C, parents, toks, doms[0])])
    assert st == native.TSS_OK
    ref, _ = O.verify_request(wo, ARCH, skips[0], toks, parents, C, O.prefill(wo, ARCH, skips[0], full[0]))
    assert_logits(res["logits"].cpu().numpy(), ref, "verify after GPU prefill")
    run.close()


@pytest.mark.parametrize("path", PATHS)
def test_all_layers_skipped_is_embedding_norm_lm_head(weights, path):
    w, wo, wg = weights
    run = make_runner(wg, n_slots=1, cap=64, path=path)
    run.set_phi({0: (1 << ARCH.n_layers) - 1})
    parents = synth.chain_parents(3)
    toks = [5, 17, 2047, 0]
    res, st = run_step(run, [synth.Request(10, parents, toks, 0)])
    assert st == native.TSS_OK
    ref, nk = O.verify_request(wo, ARCH, frozenset(range(ARCH.n_layers)), toks, parents, 10, [None] * 4)
    assert nk == {}
    assert_logits(res["logits"].cpu().numpy(), ref, "all skipped")
    for t in run.kv:
        assert torch.count_nonzero(t) == 0
    run.close()


def test_root_only_and_empty_context(weights):
    w, wo, wg = weights
    run = make_runner(wg, n_slots=2, cap=64)
    reqs = [synth.Request(0, [-1], [42], 0), synth.Request(0, synth.chain_parents(2), [1, 2, 3], 0)]
    res, st = run_step(run, reqs)
    assert st == native.TSS_OK
    gl = res["logits"].cpu().numpy()
    empty = [O.empty_kv(ARCH) for _ in range(4)]
    r0, _ = O.verify_request(wo, ARCH, frozenset(), [42], [-1], 0, empty)
    r1, _ = O.verify_request(wo, ARCH, frozenset(), [1, 2, 3], [-1, 0, 1], 0, empty)
    assert_logits(gl[:1], r0, "root only")
    assert_logits(gl[1:], r1, "empty context")
    assert int(res["accept_len"][0]) == 0 and int(res["new_ctx_len"][0]) == 1
    run.close()


@pytest.mark.parametrize("path", PATHS)
def test_speculative_sampling_chain(weights, path):
    """B=3 chains (k=4, 1, 3) at temperature 1 with Philox uniforms and with caller uniforms."""
    w, wo, wg = weights
    run = make_runner(wg, n_slots=3, cap=256, path=path)
    run.set_phi({0: O.set_to_mask({1}), 1: 0})
    ks, ctxs, doms = [4, 1, 3], [64, 33, 90], [0, 1, 0]
    reqs, kvs, skips, qs = [], [], [], []
    for b in range(3):
        skip = frozenset({1}) if doms[b] == 0 else frozenset()
        ctx = synth.uniform_ints(ctxs[b], ARCH.vocab, SEED, f"samp.ctx{b}").tolist()
        kv = O.prefill(wo, ARCH, skip, ctx)
        upload_context(run, kv, b)
        q, samp = synth.draft_probs_and_samples(ks[b] + 1, ARCH.vocab, SEED, f"samp.q{b}")
        toks = [int(synth.uniform_ints(1, ARCH.vocab, SEED, f"samp.root{b}").item())] + samp[1:]
        reqs.append(synth.Request(ctxs[b], synth.chain_parents(ks[b]), toks, doms[b], q))
        kvs.append(kv)
        skips.append(skip)
        qs.append(q)
    probs = torch.cat(qs, 0).cuda()
    counts = {"exact": 0, "flagged": 0, "slack": 0}
    for trial in range(6):
        use_unif = trial % 2 == 1
        stride = 2 * max(ks) + 1
        unif = synth.uniform01(3 * stride, SEED, f"samp.u{trial}").float().view(3, stride)
        kw = dict(mode=native.TSS_MODE_SAMPLE, temperature=1.0, draft_probs=probs, philox_seed=1234,
                  philox_offset=trial)
        if use_unif:
            kw["uniforms"] = unif.cuda()
        res, st = run_step(run, reqs, **kw)
        assert st == native.TSS_OK
        gl = res["logits"].cpu().numpy()
        off = 0
        for b, r in enumerate(reqs):
            n = len(r.parents)
            ref, _ = O.verify_request(wo, ARCH, skips[b], r.tokens, r.parents, r.ctx_len, kvs[b])
            assert_logits(gl[off:off + n], ref, f"sample request {b}")
            u = unif[b].double().numpy() if use_unif else O.philox_uniforms(1234, trial, b, ks[b])
            ga, gb = int(res["accept_len"][b]), int(res["bonus"][b])
            kind = check_sample(ref, gl[off:off + n], r.tokens, qs[b].numpy(), u, 1.0, ga, gb,
                                f"trial {trial} req {b}")
            counts[kind] += 1
            off += n
    print(f"[parity] speculative sampling ({path}): {counts}")
    assert sum(counts.values()) == 18 and counts["exact"] >= 12
    run.close()


def test_persistent_path_is_deterministic_and_close_to_multi_kernel_path(weights):
    w, wo, wg = weights
    reqs = [synth.Request(40, synth.chain_parents(4), [3, 1, 4, 1, 5], 0),
            synth.Request(17, [-1, 0, 0, 1], [7, 8, 9, 10], 1)]
    outs = {}
    for path in PATHS:
        run = make_runner(wg, n_slots=2, cap=64, path=path)
        run.set_phi({0: O.set_to_mask({3}), 1: O.set_to_mask({0})})
        for l in range(4):
            run.kv[l].copy_(synth.normal_bf16(run.kv[l].shape, SEED, f"pm{l}", 0.5).cuda())
        r1, s1 = run_step(run, reqs)
        r2, s2 = run_step(run, reqs)
        assert s1 == s2 == native.TSS_OK
        assert torch.equal(r1["logits"], r2["logits"])
        outs[path] = r1["logits"].cpu().numpy()
        run.close()
    assert np.abs(outs["persistent"] - outs["multi"]).max() < 2e-2
    assert np.abs(outs["persistent"] - outs["hybrid"]).max() < 2e-2


def test_graph_and_eager_paths_agree_bitwise(weights):
    w, wo, wg = weights
    reqs = [synth.Request(40, synth.chain_parents(4), [3, 1, 4, 1, 5], 0)]
    outs = []
    for eager in (False, True):
        os.environ["TSS_NO_GRAPH"] = "1" if eager else "0"
        try:
            run = make_runner(wg, n_slots=1, cap=64, path="multi")
        finally:
            os.environ.pop("TSS_NO_GRAPH", None)
        run.set_phi({0: O.set_to_mask({3})})
        for l in range(4):
            run.kv[l].copy_(synth.normal_bf16(run.kv[l].shape, SEED, f"ge{l}", 0.5).cuda())
        r1, _ = run_step(run, reqs)
        r2, _ = run_step(run, reqs)
        assert torch.equal(r1["logits"], r2["logits"])  # deterministic
        outs.append(r1["logits"].clone())
        run.close()
    assert torch.equal(outs[0], outs[1])


def test_host_io_matches_device_io(weights):
    w, wo, wg = weights
    run = make_runner(wg, n_slots=2, cap=64)
    for l in range(4):
        run.kv[l].copy_(synth.normal_bf16(run.kv[l].shape, SEED, f"io{l}", 0.5).cuda())
    reqs = [synth.Request(30, synth.chain_parents(3), [9, 8, 7, 6], 0), synth.Request(12, [-1, 0, 0], [1, 2, 3], 0)]
    dev, _ = run_step(run, reqs)
    hres = run.alloc_results(2, 7, host=True)
    b = run.batch(reqs, io_host=True)
    run.verify(b, hres)
    assert run.sync_status() == native.TSS_OK
    for key in ("accept_len", "bonus", "new_ctx_len", "path"):
        assert torch.equal(hres[key], dev[key].cpu())
    assert torch.equal(hres["logits"], dev["logits"].cpu())
    run.close()


def test_linear_matches_matmul(weights):
    w, wo, wg = weights
    run = make_runner(wg, n_slots=1, cap=16)
    for m, k, n in [(1, 64, 128), (6, 256, 384), (61, 512, 640), (144, 128, 256), (256, 192, 128), (17, 4096, 1024)]:
        x = synth.normal_bf16((m, k), SEED, f"lx{m}", 1.0).cuda()
        wt = synth.normal_bf16((n, k), SEED, f"lw{n}", 0.05).cuda()
        y = torch.empty((m, n), dtype=torch.float32, device="cuda")
        run.v.linear(x, wt, y)
        torch.cuda.synchronize()
        ref = x.double().cpu().numpy() @ wt.double().cpu().numpy().T
        np.testing.assert_allclose(y.cpu().numpy(), ref, rtol=1e-4, atol=1e-4, err_msg=f"{m}x{k}x{n}")
    run.close()


def test_host_validation_errors(weights):
    w, wo, wg = weights
    run = make_runner(wg, n_slots=2, cap=32)
    res = run.alloc_results(2, 8)

    def status(reqs, **kw):
        b = run.batch(reqs, **kw)
        try:
            run.verify(b, res)
            return native.TSS_OK
        except native.TssError as e:
            return e.status

    good = synth.Request(4, [-1, 0], [1, 2], 0)
    assert status([synth.Request(4, [-1, 1], [1, 2], 0)]) == native.TSS_ERR_INVALID_ARG  # parent not before child
    assert status([synth.Request(4, [0, 0], [1, 2], 0)]) == native.TSS_ERR_INVALID_ARG  # root must be -1
    assert status([synth.Request(31, [-1, 0], [1, 2], 0)]) == native.TSS_ERR_KV_CAPACITY
    assert status([good, good], slots=[1, 1]) == native.TSS_ERR_INVALID_ARG  # shared slot
    assert status([synth.Request(4, [-1, 0, 0], [1, 2, 3], 0)], mode=native.TSS_MODE_SAMPLE,
                  draft_probs=torch.ones(3, ARCH.vocab, device="cuda")) == native.TSS_ERR_INVALID_ARG  # tree
    assert status([good], mode=native.TSS_MODE_SAMPLE) == native.TSS_ERR_INVALID_ARG  # no draft probs
    with pytest.raises(native.TssError):
        run.v.set_skip_config(0, 1 << ARCH.n_layers)
    with pytest.raises(native.TssError):
        run.v.set_skip_config(-1, 0)  # domain id out of range
    # size limits: more nodes than a request may have, more rows than the context was created for,
    # more requests than its batch limit, no request at all
    big = synth.Request(0, synth.chain_parents(64), list(range(65)), 0)
    assert status([big]) == native.TSS_ERR_INVALID_ARG
    assert status([good] * 9, slots=list(range(9))) == native.TSS_ERR_INVALID_ARG
    assert status([]) == native.TSS_ERR_INVALID_ARG
    assert status([synth.Request(4, [-1, 0], [1, 2], 0)], slots=[2]) == native.TSS_ERR_INVALID_ARG  # slot range
    assert status([good], mode=native.TSS_MODE_SAMPLE, temperature=0.0,
                  draft_probs=torch.ones(2, ARCH.vocab, device="cuda")) == native.TSS_ERR_INVALID_ARG
    assert status([good]) == native.TSS_OK
    assert run.sync_status() == native.TSS_OK
    run.close()
    # more rows in one step than the context was created for
    run = make_runner(wg, n_slots=3, cap=80, max_rows=128)
    many = [synth.Request(0, synth.chain_parents(63), list(range(64)), 0) for _ in range(3)]
    b = run.batch(many)
    with pytest.raises(native.TssError) as err:
        run.verify(b, run.alloc_results(3, 192))
    assert err.value.status == native.TSS_ERR_INVALID_ARG
    run.close()


def test_device_check_reports_bad_token(weights):
    w, wo, wg = weights
    run = make_runner(wg, n_slots=1, cap=32)
    res = run.alloc_results(1, 2)
    b = run.batch([synth.Request(4, [-1, 0], [1, ARCH.vocab + 5], 0)])
    run.verify(b, res)
    assert run.sync_status() == native.TSS_ERR_DEVICE_CHECK
    assert run.sync_status() == native.TSS_OK  # cleared
    run.close()


def test_sparsity_ratio_and_active_layers(weights):
    w, wo, wg = weights
    run = make_runner(wg, n_slots=2, cap=32)
    run.set_phi({0: O.set_to_mask({1, 3}), 1: O.set_to_mask({1})})
    assert run.v.sparsity_ratio(0) == 0.5 and run.v.sparsity_ratio(5) == 0.0
    b = run.batch([synth.Request(1, [-1], [1], 0), synth.Request(1, [-1], [1], 1)])
    assert run.v.active_layer_count(b) == 3  # union: layer 1 skipped by both
    run.v.clear_skip_config(1)
    assert run.v.active_layer_count(b) == 4
    run.close()


def test_create_reports_out_of_memory_under_an_allocation_limit(weights, monkeypatch):
    """Failure injection on the host: with TSS_ALLOC_LIMIT_BYTES below what tss_create needs, the
    call returns TSS_ERR_OUT_OF_MEMORY, frees what it had allocated, and a later create without
    the limit succeeds."""
    _, _, wg = weights
    monkeypatch.setenv("TSS_ALLOC_LIMIT_BYTES", str(1 << 20))
    with pytest.raises(native.TssError) as err:
        native.Verifier(wg, ARCH, max_batch=1, max_rows=8, max_nodes=8)
    assert err.value.status == native.TSS_ERR_OUT_OF_MEMORY
    assert "TSS_ALLOC_LIMIT_BYTES" in str(err.value)
    monkeypatch.delenv("TSS_ALLOC_LIMIT_BYTES")
    v = native.Verifier(wg, ARCH, max_batch=1, max_rows=8, max_nodes=8)
    v.close()



@pytest.mark.parametrize("path", ["persistent", "hybrid"])
def test_bounded_wait_times_out_and_the_context_recovers(weights, path, monkeypatch):
    """Failure injection without a GPU fault: with a 200 ms wait limit, a step that withholds one
    dataflow flag (tss_inject_timeout) ends with TSS_ERR_TIMEOUT from the bounded waits, and the
    next step on the same context runs normally and matches the oracle."""
    w, wo, wg = weights
    monkeypatch.setenv("TSS_WAIT_LIMIT_MS", "200")
    run = make_runner(wg, n_slots=1, cap=128, path=path)
    skip = frozenset({2})
    run.set_phi({0: O.set_to_mask(skip)})
    ctx = synth.uniform_ints(40, ARCH.vocab, SEED, "to.ctx").tolist()
    kv = O.prefill(wo, ARCH, skip, ctx)
    upload_context(run, kv, 0)
    parents = synth.chain_parents(4)
    toks = synth.draft_tokens(parents, ARCH.vocab, SEED, "to.tok")
    req = synth.Request(len(ctx), parents, toks, 0)
    run.v.inject_timeout(1)
    _, st = run_step(run, [req])
    assert st == native.TSS_ERR_TIMEOUT
    assert run.sync_status() == native.TSS_OK  # reported once, then cleared
    for _ in range(2):
        res, st = run_step(run, [req])
        assert st == native.TSS_OK
        ref, _ = O.verify_request(wo, ARCH, skip, toks, parents, len(ctx), kv)
        assert_logits(res["logits"].cpu().numpy(), ref, f"after a timeout ({path})")
    run.close()


def test_device_philox_matches_the_oracle_generator():
    """tss_philox_uniforms (the device generator the acceptance kernels draw from) against the
    oracle's Philox4x32-10 on 10^6 counters: all four output words and the uniforms, for seed and
    offset words beyond 2^32."""
    from oracle import philox as P
    from paper_2609_26100_gb300 import build
    build.build()
    n_req, n_slots = 1000, 334
    for seed, offset in [(42, 3), ((7 << 32) | 0x9E3779B9, (1 << 40) + 5), (0xFFFFFFFFFFFFFFFF, 0xFFFFFFFF00000001)]:
        words = torch.empty((n_req, n_slots, 4), dtype=torch.int32, device="cuda")
        unif = torch.empty((n_req, n_slots), dtype=torch.float32, device="cuda")
        native.philox_uniforms(seed, offset, words=words, uniforms=unif)
        torch.cuda.synchronize()
        got = words.cpu().numpy().view(np.uint32)
        req, slot = np.meshgrid(np.arange(n_req, dtype=np.uint64), np.arange(n_slots, dtype=np.uint64), indexing="ij")
        ctr = np.stack([slot, req, np.full_like(req, offset & 0xFFFFFFFF), np.full_like(req, offset >> 32)], axis=-1)
        ref = P.philox4x32_10(ctr, np.array([seed & 0xFFFFFFFF, seed >> 32], dtype=np.uint64))
        assert np.array_equal(got, ref), f"seed {seed:#x} offset {offset:#x}"
        assert np.array_equal(unif.cpu().numpy().astype(np.float64), P.to_uniform24(ref[..., 0]))
    # the acceptance's own uniforms for a request are this stream's first 2k+1 slots
    assert np.array_equal(O.philox_uniforms(42, 3, 7, 5), P.to_uniform24(
        P.philox4x32_10(np.stack([np.arange(11, dtype=np.uint64), np.full(11, 7, np.uint64), np.full(11, 3, np.uint64),
                                  np.zeros(11, np.uint64)], -1), np.array([42, 0], np.uint64))[:, 0]))


def test_search_with_measured_verification_latency(weights):
    """Algorithm 1 with the verification cost C_d(S) measured by tss_verify on the GPU (tiny model,
    every subset of its 4 layers up to depth 2, synthetic acceptance and metric): the dense step
    is slower than every 2-layer skip, and the chosen set is feasible."""
    w, wo, wg = weights
    from paper_2609_26100_gb300 import search
    run = make_runner(wg, n_slots=1, cap=128)
    reqs = [synth.Request(64, synth.chain_parents(4), [1, 2, 3, 4, 5], 0)]
    cost = search.latency_cost(run, reqs, steps=20)
    res = search.breadth_search(ARCH.n_layers, search.combine(search.SyntheticObjective(ARCH.n_layers, 7), cost), 2,
                                0.3, 0.05, 0.3, 0.05)
    lat = {s: e.cost for s, e in res.log}
    print(f"[search] latency us by skip set: { {str(s): round(v, 1) for s, v in lat.items()} }")
    assert all(lat[()] > v for s, v in lat.items() if len(s) == 2)
    assert res.best in [s for k in res.feasible for s in res.feasible[k]]
    assert run.sync_status() == native.TSS_OK
    run.close()


WIDE = (8, 4, 3, 2, 2, 1, 1, 1)  # a wide static draft tree (SAMD / token-recycling style), beyond 64 nodes


@pytest.mark.parametrize("path", PATHS)
def test_blocks_beyond_64_rows(weights, path):
    """A 127-node wide draft tree (128 rows) with a planted greedy path and a 99-draft chain (100
    rows) in one 228-row step: logits of every row, the tree walk and the chain's acceptance, the
    tree's KV compacted to its path, and a skipped layer left untouched.  Blocks over 64 rows take
    the separate attention kernel's wide variant (two-word ancestor mask, eight 16-row query tiles)
    on every path."""
    w, wo, wg = weights
    run = make_runner(wg, n_slots=2, cap=400, path=path, max_nodes=128)
    phi = {0: O.set_to_mask({2}), 1: 0}
    run.set_phi(phi)
    sentinel = 7.0
    for t in run.kv:
        t.fill_(sentinel)
    skips = [frozenset({2}), frozenset()]
    ctxs = [150, 90]
    kvs = []
    for b in range(2):
        kv = O.prefill(wo, ARCH, skips[b], synth.uniform_ints(ctxs[b], ARCH.vocab, SEED, f"wide.ctx{b}").tolist())
        upload_context(run, kv, b)
        kvs.append(kv)
    tree = synth.eagle_tree(127, WIDE)
    assert len(tree) == 128 and max(synth.depths_of(tree)) >= 5
    toks = synth.draft_tokens(tree, ARCH.vocab, SEED, "wide.tok")
    toks[0] = 23
    greedy = greedy_ar(wo, skips[0], kvs[0], toks[0], ctxs[0], 5)
    ch = O.children_of(tree)
    cur = 0
    for rank, g in zip((3, 0, 0, 0, 0), greedy):  # the path's first node is row 110 of the block
        if len(ch[cur]) <= rank:
            break
        nxt = ch[cur][rank]
        for sib in ch[cur]:
            if toks[sib] == g:
                toks[sib] = (g + 7) % ARCH.vocab
        toks[nxt] = g
        cur = nxt
    chain = synth.chain_parents(99)
    ctoks = synth.draft_tokens(chain, ARCH.vocab, SEED, "wide.chain")
    reqs = [synth.Request(ctxs[0], tree, toks, 0), synth.Request(ctxs[1], chain, ctoks, 1)]
    res, st = run_step(run, reqs)
    assert st == native.TSS_OK
    gl = res["logits"].cpu().numpy()
    ref_t, nk_t = O.verify_request(wo, ARCH, skips[0], toks, tree, ctxs[0], kvs[0])
    ref_c, _ = O.verify_request(wo, ARCH, skips[1], ctoks, chain, ctxs[1], kvs[1])
    assert_logits(gl[:128], ref_t, "127-node tree")
    assert_logits(gl[128:], ref_c, "100-row chain")
    for b, (ref, tk, par) in enumerate([(ref_t, toks, tree), (ref_c, ctoks, chain)]):
        a, bonus, pth = O.greedy_accept(ref, tk, par)
        ga, gb = int(res["accept_len"][b]), int(res["bonus"][b])
        gp = gpu_path(res, b, ga)
        if O.greedy_flagged(ref, pth):
            assert greedy_valid(ref, tk, par, gp, gb)
        else:
            assert (ga, gb, gp) == (a, bonus, pth)
            if b == 0:
                assert a >= 1 and gp[1] > 64
    ga = int(res["accept_len"][0])
    gp = gpu_path(res, 0, ga)
    C = ctxs[0]
    for l in nk_t:
        gk = run.kv[l][0, 0, :, C:C + ga + 1].float().cpu().numpy()
        np.testing.assert_allclose(gk, np.transpose(O.compact_block_rows(nk_t[l][0], gp), (1, 0, 2)), atol=3e-2,
                                   rtol=2e-2)
    assert bool((run.kv[2][0] == sentinel).all())  # request 0 skips layer 2
    run.close()


@pytest.mark.parametrize("mode", ["greedy", "sample"])
def test_grouped_verification_equals_mixed_step_and_oracle(weights, mode):
    """tss_verify_grouped on a mixed batch of four requests (two skip sets, one dense domain and one
    unconfigured domain, which share the dense path): three groups, the one with the most skipped
    layers first; every request's logits, acceptance and path equal the oracle's and the mixed
    step's (sampling: the same Philox uniforms per request), and the groups' events complete in
    order."""
    w, wo, wg = weights
    phi = {0: O.set_to_mask({2}), 1: O.set_to_mask({0, 3}), 2: 0}
    doms = [2, 1, 0, 7]
    ctxs = [60, 33, 90, 12]
    ks = [3, 4, 2, 5]
    run = make_runner(wg, n_slots=4, cap=160)
    run.set_phi(phi)
    reqs, kvs, skips, qs = [], [], [], []
    for b in range(4):
        skip = O.skip_set({d: O.mask_to_set(m) for d, m in phi.items()}, doms[b])
        kv = O.prefill(wo, ARCH, skip, synth.uniform_ints(ctxs[b], ARCH.vocab, SEED, f"grp.ctx{b}").tolist())
        upload_context(run, kv, b)
        q, samp = synth.draft_probs_and_samples(ks[b] + 1, ARCH.vocab, SEED, f"grp.q{b}")
        toks = [int(synth.uniform_ints(1, ARCH.vocab, SEED, f"grp.root{b}").item())] + samp[1:]
        reqs.append(synth.Request(ctxs[b], synth.chain_parents(ks[b]), toks, doms[b], q))
        kvs.append(kv)
        skips.append(skip)
        qs.append(q)
    kw = {}
    if mode == "sample":
        kw = dict(mode=native.TSS_MODE_SAMPLE, temperature=1.0, draft_probs=torch.cat(qs, 0).cuda(), philox_seed=77,
                  philox_offset=5)
    rows = sum(len(r.parents) for r in reqs)
    mixed = run.alloc_results(4, rows)
    run.verify(run.batch(reqs, **kw), mixed)
    grouped = run.alloc_results(4, rows)
    events = [torch.cuda.Event(enable_timing=True) for _ in range(4)]
    n_groups = run.verify_grouped(run.batch(reqs, **kw), grouped, events=events)
    assert run.sync_status() == native.TSS_OK
    torch.cuda.synchronize()
    assert n_groups == 3
    assert events[0].elapsed_time(events[1]) > 0 and events[1].elapsed_time(events[2]) > 0
    for key in ("accept_len", "bonus", "new_ctx_len", "path"):
        assert torch.equal(grouped[key], mixed[key]), key
    gl = grouped["logits"].cpu().numpy()
    assert np.abs(gl - mixed["logits"].cpu().numpy()).max() < 1e-3
    off = 0
    for b, r in enumerate(reqs):
        n = len(r.parents)
        ref, _ = O.verify_request(wo, ARCH, skips[b], r.tokens, r.parents, r.ctx_len, kvs[b])
        assert_logits(gl[off:off + n], ref, f"grouped request {b}")
        ga, gb = int(grouped["accept_len"][b]), int(grouped["bonus"][b])
        if mode == "greedy":
            a, bonus, pth = O.greedy_accept(ref, r.tokens, r.parents)
            if not O.greedy_flagged(ref, pth):
                assert (ga, gb) == (a, bonus)
        else:
            u = O.philox_uniforms(77, 5, b, ks[b])
            check_sample(ref, gl[off:off + n], r.tokens, qs[b].numpy(), u, 1.0, ga, gb, f"grouped request {b}")
        off += n
    run.close()
