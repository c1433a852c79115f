"""GPU parity at the full sizes of the 7B / 13B workloads, in the configuration bench.py times
(TssRunner.for_workload, default persistent path): the CUDA path through the C ABI against the
CPU oracle on sampled requests, which the oracle recomputes one by one with every layer's
weights and context KV regenerated from the seeded generators on access (a 7B layer is 0.8 GB
in fp32, so nothing is cached), plus properties that hold at any size for the other requests.

The seeded generators are elementwise integer hashes, so generating on the GPU and copying to
the host gives the CPU generator's values; test_synth_device_matches_host pins that."""
import numpy as np
import pytest
import torch

from oracle import tss_oracle as O
from paper_2609_26100_gb300 import native, synth
from tests.parity_util import assert_logits, greedy_valid, gpu_path

pytestmark = [pytest.mark.gpu, pytest.mark.slow]


@pytest.fixture(scope="module", autouse=True)
def _library():
    from paper_2609_26100_gb300 import build
    build.build()
    yield
    torch.cuda.empty_cache()


def _host_budget_bytes():
    """Host memory the tests may use for cached oracle layers: 40 % of MemAvailable."""
    try:
        with open("/proc/meminfo") as f:
            for ln in f:
                if ln.startswith("MemAvailable:"):
                    return int(ln.split()[1]) * 1024 * 0.4
    except OSError:
        pass
    return 0


class LazyLayers:
    """weights["layers"][l] for the oracle: layer l regenerated (seeded) and copied to host fp32;
    kept for later accesses while the host memory budget allows."""

    def __init__(self, arch, seed):
        self.arch, self.seed = arch, seed
        self.cache, self.budget = {}, _host_budget_bytes()

    def __getitem__(self, l):
        if l in self.cache:
            return self.cache[l]
        lw = synth.make_layer(self.arch, l, self.seed, device="cuda")
        out = {k: v.float().cpu().numpy() for k, v in lw.items()}
        size = sum(v.nbytes for v in out.values())
        if size * (len(self.cache) + 1) <= self.budget:
            self.cache[l] = out
        return out


class LazyKV:
    """kv[l] for the oracle: request `req`'s synthetic context KV of layer l, (K [H,C,D], V)."""

    def __init__(self, arch, seed, req, ctx):
        self.arch, self.seed, self.req, self.ctx = arch, seed, req, ctx

    def __getitem__(self, l):
        blk = synth.kv_block(self.arch, l, self.req, self.ctx, self.seed, device="cuda").float().cpu().numpy()
        return blk[0], blk[1]


def oracle_weights(w):
    g = synth.make_weights(w.arch, w.seed, device="cuda", layers=[])
    out = {"embed": g["embed"].float().cpu().numpy(), "lm_head": g["lm_head"].float().cpu().numpy(),
           "final_norm": g["final_norm"].float().cpu().numpy(), "layers": LazyLayers(w.arch, w.seed)}
    del g
    torch.cuda.empty_cache()
    return out


def skip_of(w, b):
    return frozenset(synth.layers_of(w.skip_mask(b)))


class AppendedKV:
    """kv[l] for the oracle in a lockstep run: request `req`'s synthetic context of ctx0 tokens plus
    the rows appended by the accepted paths of earlier steps (K/V [H, n, D] per layer)."""

    def __init__(self, arch, seed, req, ctx0):
        self.base = LazyKV(arch, seed, req, ctx0)
        self.rows = {}

    def append(self, new_kv, path):
        for l, (k, v) in new_kv.items():
            kk, vv = np.transpose(k[path], (1, 0, 2)), np.transpose(v[path], (1, 0, 2))
            if l in self.rows:
                kk = np.concatenate([self.rows[l][0], kk], axis=1)
                vv = np.concatenate([self.rows[l][1], vv], axis=1)
            self.rows[l] = (kk, vv)

    def __getitem__(self, l):
        k, v = self.base[l]
        if l in self.rows:
            k = np.concatenate([k, self.rows[l][0]], axis=1)
            v = np.concatenate([v, self.rows[l][1]], axis=1)
        return k, v


def oracle_request(wo, w, b, tokens=None):
    r = w.requests[b]
    toks = r.tokens if tokens is None else tokens
    return O.verify_request(wo, w.arch, skip_of(w, b), toks, r.parents, r.ctx_len,
                            LazyKV(w.arch, w.seed, b, r.ctx_len))


def run_step(run, reqs, logits=True, **kw):
    res = run.alloc_results(len(reqs), sum(len(r.parents) for r in reqs), logits=logits)
    run.verify(run.batch(reqs, **kw), res)
    st = run.sync_status()
    torch.cuda.synchronize()
    assert st == native.TSS_OK, f"device status {st}"
    return res


def check_greedy(ref, toks, parents, res, b):
    """accept_len, bonus and path equal the oracle's unless the step is flagged (near-tie)."""
    a, bonus, path = O.greedy_accept(ref, toks, parents)
    ga, gb = int(res["accept_len"][b]), int(res["bonus"][b])
    gp = gpu_path(res, b, ga)
    if O.greedy_flagged(ref, path):
        assert greedy_valid(ref, toks, parents, gp, gb)
        return None
    assert (ga, gb, gp) == (a, bonus, path)
    return a


def test_synth_device_matches_host():
    """The generators give identical values on the GPU and on the host (weights, KV, draws)."""
    a = synth.TINY
    for l in (0, 3):
        hc, hg = synth.make_layer(a, l, 42), synth.make_layer(a, l, 42, device="cuda")
        for k in hc:
            assert torch.equal(hc[k], hg[k].cpu()), k
    assert torch.equal(synth.kv_block(a, 1, 2, 77, 42), synth.kv_block(a, 1, 2, 77, 42, device="cuda").cpu())
    big = synth.LLAMA2_7B
    t_host = synth.normal_bf16((1024, big.d_model), 42, "probe", 0.02)
    t_dev = synth.normal_bf16((1024, big.d_model), 42, "probe", 0.02, device="cuda")
    assert torch.equal(t_host, t_dev.cpu())


def test_7b_chain_full_size():
    """7B, ctx 1024, chain k=5, skip {20,24,27,30} and dense: logits of every row, greedy
    acceptance, and a step whose first draft is the oracle's greedy token (accept_len >= 1)."""
    w = synth.workload_7b_chain()
    w.phi[1] = 0  # the dense configuration as a second domain
    from paper_2609_26100_gb300.runner import TssRunner
    run = TssRunner.for_workload(synth.workload_7b_chain(mask_layers=()))  # every layer's weights and KV
    run.set_phi(w.phi)
    wo = oracle_weights(w)
    r = w.requests[0]
    # step 1: the workload's random draft under the skip set
    res = run_step(run, w.requests)
    ref, _ = oracle_request(wo, w, 0)
    assert_logits(res["logits"].cpu().numpy(), ref, "7b chain skip4")
    check_greedy(ref, r.tokens, r.parents, res, 0)
    # step 2: first draft = the oracle's greedy token after the root
    toks = list(r.tokens)
    toks[1] = O.argmax_lowest(ref[0])
    req2 = synth.Request(r.ctx_len, r.parents, toks, 0)
    res2 = run_step(run, [req2])
    ref2, _ = oracle_request(wo, w, 0, tokens=toks)
    assert_logits(res2["logits"].cpu().numpy(), ref2, "7b chain skip4, greedy first draft")
    a2 = check_greedy(ref2, toks, r.parents, res2, 0)
    assert a2 is None or a2 >= 1
    # step 3: the same block with the dense configuration (domain 1)
    w_dense = synth.workload_7b_chain(mask_layers=())
    res3 = run_step(run, [synth.Request(r.ctx_len, r.parents, r.tokens, 1)])
    ref3, _ = oracle_request(wo, w_dense, 0)
    assert_logits(res3["logits"].cpu().numpy(), ref3, "7b chain dense")
    check_greedy(ref3, r.tokens, r.parents, res3, 0)
    run.close()


def test_7b_chain_lockstep_steps():
    """Four consecutive 7B chain steps (ctx 1024 growing, k=5, skip {20,24,27,30}) in lockstep with
    the oracle: each step's logits, greedy acceptance and appended KV rows; steps 1 and 3 start
    with the oracle's greedy token (accept_len >= 1); after each step the oracle's accepted rows
    replace the GPU's in the cache, and the next root is the oracle's bonus token."""
    w = synth.workload_7b_chain()
    from paper_2609_26100_gb300.runner import TssRunner
    run = TssRunner.for_workload(w, extra_cap=4 * 6)
    a_ = w.arch
    r = w.requests[0]
    wo = oracle_weights(w)
    skip = skip_of(w, 0)
    kv = AppendedKV(a_, w.seed, 0, r.ctx_len)
    C, root = r.ctx_len, r.tokens[0]
    exact = flagged = 0
    for step in range(4):
        parents = r.parents
        toks = [root] + synth.draft_tokens(parents, a_.vocab, w.seed, f"full.lock{step}")[1:]
        if step % 2 == 1:
            ref0, _ = O.verify_request(wo, a_, skip, toks, parents, C, kv)
            toks[1] = O.argmax_lowest(ref0[0])
        res = run_step(run, [synth.Request(C, parents, toks, 0)])
        ref, nk = O.verify_request(wo, a_, skip, toks, parents, C, kv)
        assert_logits(res["logits"].cpu().numpy(), ref, f"7b chain lockstep step {step}")
        a, bonus, path = O.greedy_accept(ref, toks, parents)
        got = check_greedy(ref, toks, parents, res, 0)
        if got is None:
            flagged += 1
        else:
            exact += 1
            if step % 2 == 1:
                assert got >= 1
        for l in synth.seeded_subset(sorted(nk), 2, w.seed, f"full.lock.layers{step}"):
            gk = run.kv[l][0, 0, :, C:C + len(parents)].float().cpu().numpy()
            np.testing.assert_allclose(gk, np.transpose(nk[l][0], (1, 0, 2)), atol=5e-2, rtol=3e-2)
        kv.append(nk, path)  # lockstep on the oracle's state
        for l in nk:
            run.write_kv(l, 0, torch.from_numpy(np.ascontiguousarray(np.transpose(nk[l][0][path], (1, 0, 2)))),
                         torch.from_numpy(np.ascontiguousarray(np.transpose(nk[l][1][path], (1, 0, 2)))), pos0=C)
        C += 1 + a
        root = bonus
    print(f"[parity] 7b chain lockstep: {exact} exact, {flagged} flagged")
    run.close()


def test_7b_tree_full_size():
    """7B, ctx 2048, 60-node tree, 6 skipped layers: logits of all 61 rows, greedy longest
    matching path with a planted first step, and the KV compacted to that path."""
    w = synth.workload_7b_tree()
    from paper_2609_26100_gb300.runner import TssRunner
    run = TssRunner.for_workload(w)
    wo = oracle_weights(w)
    r = w.requests[0]
    ref0, _ = oracle_request(wo, w, 0)
    # plant the root's greedy token on its second child (siblings keep distinct tokens)
    toks = list(r.tokens)
    ch = O.children_of(r.parents)
    g = O.argmax_lowest(ref0[0])
    for sib in ch[0]:
        if toks[sib] == g:
            toks[sib] = (g + 7) % w.arch.vocab
    toks[ch[0][1]] = g
    req = synth.Request(r.ctx_len, r.parents, toks, 0)
    res = run_step(run, [req])
    ref, nk = oracle_request(wo, w, 0, tokens=toks)
    assert_logits(res["logits"].cpu().numpy(), ref, "7b tree")
    a = check_greedy(ref, toks, r.parents, res, 0)
    assert a is None or a >= 1
    ga = int(res["accept_len"][0])
    gp = gpu_path(res, 0, ga)
    C = r.ctx_len
    assert int(res["new_ctx_len"][0]) == C + 1 + ga
    for l in synth.seeded_subset(sorted(nk), 3, w.seed, "full.tree.layers"):
        comp_k = O.compact_block_rows(nk[l][0], gp)
        comp_v = O.compact_block_rows(nk[l][1], gp)
        gk = run.kv[l][0, 0, :, C:C + ga + 1].float().cpu().numpy()
        gv = run.kv[l][0, 1, :, C:C + ga + 1].float().cpu().numpy()
        np.testing.assert_allclose(gk, np.transpose(comp_k, (1, 0, 2)), atol=5e-2, rtol=3e-2)
        np.testing.assert_allclose(gv, np.transpose(comp_v, (1, 0, 2)), atol=5e-2, rtol=3e-2)
    for l in synth.layers_of(w.skip_mask(0)):
        assert run.kv[l] is None  # a layer no request runs has no cache and is never touched
    run.close()


def test_13b_mixed_sampling_full_size():
    """13B, B=8, ctx ~U[512,4096], 6 domains, chain k=5, speculative sampling at T=1 with
    Philox uniforms: every request recomputed by the oracle (logits, accept decisions and drawn
    tokens, exact wherever the measured logit error moves no decision) and its outputs in range."""
    from tests.parity_util import check_sample
    w = synth.workload_13b_mixed()
    from paper_2609_26100_gb300.runner import TssRunner
    run = TssRunner.for_workload(w)
    probs = torch.cat([r.draft_probs for r in w.requests], 0).cuda()
    res = run_step(run, w.requests, mode=native.TSS_MODE_SAMPLE, temperature=w.temperature, draft_probs=probs,
                   philox_seed=w.seed, philox_offset=3)
    gl = res["logits"].cpu().numpy()
    offs = np.cumsum([0] + [len(r.parents) for r in w.requests])
    for b, r in enumerate(w.requests):
        k = len(r.parents) - 1
        ga = int(res["accept_len"][b])
        assert 0 <= ga <= k and 0 <= int(res["bonus"][b]) < w.arch.vocab
        assert int(res["new_ctx_len"][b]) == r.ctx_len + 1 + ga
    run.close()
    torch.cuda.empty_cache()
    wo = oracle_weights(w)
    B = len(w.requests)
    kvs = [LazyKV(w.arch, w.seed, b, r.ctx_len) for b, r in enumerate(w.requests)]
    refs = O.verify_requests(wo, w.arch, [skip_of(w, b) for b in range(B)],
                             [(r.tokens, r.parents, r.ctx_len) for r in w.requests], lambda b, l: kvs[b][l])
    counts = {"exact": 0, "flagged": 0, "slack": 0}
    for b, r in enumerate(w.requests):
        ref = refs[b][0]
        assert_logits(gl[offs[b]:offs[b + 1]], ref, f"13b request {b}")
        u = O.philox_uniforms(w.seed, 3, b, len(r.parents) - 1)
        kind = check_sample(ref, gl[offs[b]:offs[b + 1]], r.tokens, r.draft_probs.numpy(), u, w.temperature,
                            int(res["accept_len"][b]), int(res["bonus"][b]), f"13b request {b}")
        counts[kind] += 1
    print(f"[parity] 13b speculative sampling, 8 requests: {counts}")


def test_7b_long_context_full_size():
    """7B KV-bound regime: B=16, ctx 16384, chain k=8, 8 skipped layers.  Three or four seeded
    requests are recomputed by the oracle; all requests: outputs in range, context KV untouched,
    and a repeated step is bitwise identical."""
    w = synth.workload_7b_long()
    from paper_2609_26100_gb300.runner import TssRunner
    run = TssRunner.for_workload(w)
    res = run_step(run, w.requests)
    gl = res["logits"].cpu().numpy()
    res_again = run_step(run, w.requests)
    assert np.array_equal(gl, res_again["logits"].cpu().numpy())
    for key in ("accept_len", "bonus", "path", "new_ctx_len"):
        assert torch.equal(res[key], res_again[key])
    k = len(w.requests[0].parents) - 1
    for b, r in enumerate(w.requests):
        ga = int(res["accept_len"][b])
        assert 0 <= ga <= k and int(res["new_ctx_len"][b]) == r.ctx_len + 1 + ga
    # the context part of a sampled layer's cache is what fill_synthetic wrote
    l = w.active_union()[len(w.active_union()) // 2]
    b = int(synth.uniform_ints(1, len(w.requests), w.seed, "full.long.req").item())
    ctx = w.requests[b].ctx_len
    assert torch.equal(run.kv[l][b, :, :, :ctx], synth.kv_block(w.arch, l, b, ctx, w.seed, device="cuda"))
    run.close()
    torch.cuda.empty_cache()
    wo = oracle_weights(w)
    picks = sorted({b} | set(synth.seeded_subset(list(range(len(w.requests))), 3, w.seed, "full.long.reqs")))
    kvs = {q: LazyKV(w.arch, w.seed, q, w.requests[q].ctx_len) for q in picks}
    refs = O.verify_requests(wo, w.arch, [skip_of(w, q) for q in picks],
                             [(w.requests[q].tokens, w.requests[q].parents, w.requests[q].ctx_len) for q in picks],
                             lambda i, l: kvs[picks[i]][l])
    n = len(w.requests[0].parents)
    for i, q in enumerate(picks):
        ref = refs[i][0]
        assert_logits(gl[q * n:(q + 1) * n], ref, f"7b long request {q}")
        check_greedy(ref, w.requests[q].tokens, w.requests[q].parents, res, q)


def test_7b_prefill_full_size():
    """The compute-bound prefill at 7B width (tokens-tiled tcgen05 GEMMs, causal tcgen05 attention):
    a 130-token prompt appended to request 0's synthetic 1024-token context under the 7B chain's
    skip set {20,24,27,30}; the K/V rows of every active layer against the oracle's (the same
    prompt as a chain block over the same context), the skipped layers untouched, and a
    verification step on top of the GPU-filled cache against the oracle."""
    w = synth.workload_7b_chain()
    from paper_2609_26100_gb300.runner import TssRunner
    n_new = 130
    run = TssRunner.for_workload(w, extra_cap=n_new + 8)
    a_ = w.arch
    r = w.requests[0]
    wo = oracle_weights(w)
    skip = skip_of(w, 0)
    C0 = r.ctx_len
    prompt = synth.uniform_ints(n_new, a_.vocab, w.seed, "full.prefill").tolist()
    run.prefill([prompt], [C0], [0])
    assert run.sync_status() == native.TSS_OK
    torch.cuda.synchronize()
    parents = [-1] + list(range(n_new - 1))
    ref_logits, new_kv = O.verify_request(wo, a_, skip, prompt, parents, C0, LazyKV(a_, w.seed, 0, C0))
    for l in range(a_.n_layers):
        if l in skip:
            assert run.kv[l] is None  # no request runs it: not even allocated
            continue
        gk = run.kv[l][0, 0, :, C0:C0 + n_new].float().cpu().numpy()
        gv = run.kv[l][0, 1, :, C0:C0 + n_new].float().cpu().numpy()
        k_ref, v_ref = np.transpose(new_kv[l][0], (1, 0, 2)), np.transpose(new_kv[l][1], (1, 0, 2))
        np.testing.assert_allclose(gk, k_ref, atol=6e-2, rtol=3e-2, err_msg=f"K layer {l}")
        np.testing.assert_allclose(gv, v_ref, atol=6e-2, rtol=3e-2, err_msg=f"V layer {l}")
        assert float(np.abs(gk - k_ref).mean()) < 4e-3, f"K layer {l}"
    # a verification step on the GPU-filled cache (context C0 + n_new)
    kv = AppendedKV(a_, w.seed, 0, C0)
    kv.append(new_kv, list(range(n_new)))
    toks = synth.draft_tokens(r.parents, a_.vocab, w.seed, "full.after_prefill")
    res = run_step(run, [synth.Request(C0 + n_new, r.parents, toks, 0)])
    ref, _ = O.verify_request(wo, a_, skip, toks, r.parents, C0 + n_new, kv)
    assert_logits(res["logits"].cpu().numpy(), ref, "7b verify after the tcgen05 prefill")
    run.close()
