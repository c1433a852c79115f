"""GPU parity of the tcgen05 attention kernel (draft blocks of at most 16 rows, head_dim 128):
the whole verification step through the C ABI against the CPU oracle, on a small decoder with
128-dimensional heads (3 layers, d 256, 2 heads x 128, MLP 688, vocab 2048), in both plans that
run a separate attention kernel -- the persistent kernel's long-context plan ("hybrid": fp16 q
split into bf16 hi + lo, P as hi + lo) and the kernel-per-operation path ("multi": bf16).

The work split cuts every (request, head) item's 128-key tiles into one range per CTA, so these
cases cover: items split over many CTAs with their partials merged (few tiles in all), CTAs that
cover several items (more tiles than SMs), contexts whose block ends exactly on a tile boundary,
a 16-node tree (ancestor mask), single-row blocks, requests that skip a layer, and cache rows past
each request's keys holding NaN (they must neither enter a score nor meet a nonzero weight)."""
import os

import numpy as np
import pytest
import torch

from oracle import tss_oracle as O
from paper_2609_26100_gb300 import native, synth
from tests.conftest import oracle_weights
from tests.parity_util import assert_logits, greedy_valid, gpu_path, to_device_weights

pytestmark = pytest.mark.gpu

ARCH = synth.Arch(n_layers=3, d_model=256, n_heads=2, head_dim=128, d_mlp=688, vocab=2048)
SEED = synth.DEFAULT_SEED
PATHS = ["hybrid", "multi"]
TC, NARROW = 1, 0  # tss_attention_kernel values


@pytest.fixture(scope="module")
def weights():
    from paper_2609_26100_gb300 import build
    build.build()
    w = synth.make_weights(ARCH)
    return oracle_weights(w), to_device_weights(w)


def make_runner(wg, n_slots, cap, path, tc=True):
    from paper_2609_26100_gb300.runner import TssRunner
    env = {"TSS_PATH": "persistent" if path == "hybrid" else "multi", "TSS_ATTN": "external",
           "TSS_ATTN_TC": "1" if tc else "0"}
    os.environ.update(env)
    try:
        return TssRunner(ARCH, wg, n_slots=n_slots, kv_cap=cap, max_batch=8, max_nodes=16)
    finally:
        for k in env:
            os.environ.pop(k, None)


def chain(ctx, k, tag, domain=0):
    parents = synth.chain_parents(k)
    return synth.Request(ctx, parents, synth.draft_tokens(parents, ARCH.vocab, SEED, tag), domain)


def tree16(ctx, tag, domain=0):
    parents = synth.eagle_tree(15, (3, 2, 2, 1))
    return synth.Request(ctx, parents, synth.draft_tokens(parents, ARCH.vocab, SEED, tag), domain)


class Case:
    """Requests with synthetic context KV in the runner's cache (every other row NaN) and the
    oracle's copy of it."""

    def __init__(self, run, reqs, phi):
        self.run, self.reqs, self.phi = run, reqs, phi
        self.skips = [O.mask_to_set(phi.get(r.domain, 0)) for r in reqs]
        run.set_phi(phi)
        for t in run.kv:
            if t is not None:
                t.fill_(float("nan"))
        self.kv = {}
        for b, r in enumerate(reqs):
            for l in range(ARCH.n_layers):
                if l in self.skips[b]:
                    continue
                blk = synth.kv_block(ARCH, l, b, r.ctx_len, SEED, device="cuda")
                run.kv[l][b, :, :, :r.ctx_len] = blk
                f = blk.float().cpu().numpy()
                self.kv[(b, l)] = (f[0], f[1])

    def step(self):
        depth = max(max(synth.depths_of(r.parents)) for r in self.reqs)
        res = self.run.alloc_results(len(self.reqs), sum(len(r.parents) for r in self.reqs),
                                     path_stride=max(64, depth + 1))
        self.run.verify(self.run.batch(self.reqs), res)
        st = self.run.sync_status()
        torch.cuda.synchronize()
        assert st == native.TSS_OK, f"device status {st}"
        return res

    def check(self, wo, res, what):
        refs = O.verify_requests(wo, ARCH, self.skips, [(r.tokens, r.parents, r.ctx_len) for r in self.reqs],
                                 lambda b, l: self.kv[(b, l)])
        gl = res["logits"].cpu().numpy()
        row = 0
        for b, (r, (ref, nk)) in enumerate(zip(self.reqs, refs)):
            n = len(r.parents)
            assert_logits(gl[row:row + n], ref, f"{what} request {b}")
            row += n
            a, bonus, path = O.greedy_accept(ref, r.tokens, r.parents)
            ga, gb = int(res["accept_len"][b]), int(res["bonus"][b])
            gp = gpu_path(res, b, ga)
            if O.greedy_flagged(ref, path):
                assert greedy_valid(ref, r.tokens, r.parents, gp, gb)
            else:
                assert (ga, gb, gp) == (a, bonus, path), f"{what} request {b}"
            # the block's K/V rows appended in every layer the request runs (before compaction they
            # sit at ctx .. ctx + n; the accepted path is then moved to ctx ..)
            for l, (k_new, _) in nk.items():
                got = self.run.kv[l][b, 0, :, r.ctx_len:r.ctx_len + 1].float().cpu().numpy()
                np.testing.assert_allclose(got[:, 0], k_new[0], atol=3e-2, rtol=2e-2)
        return refs


@pytest.mark.parametrize("path", PATHS)
def test_tc_items_split_over_many_ctas(weights, path):
    """Four requests, 56 tiles per layer: every CTA holds at most one tile and each item's
    partials are merged by the last of up to 16 CTAs.  Request 1 (a 16-node tree whose 128 keys
    fill one tile exactly) skips layer 1; request 2 is a single row (384 keys, three full tiles)."""
    wo, wg = weights
    reqs = [chain(1000, 5, "tc.a0"), tree16(112, "tc.a1", domain=1), chain(383, 0, "tc.a2"),
            chain(2000, 8, "tc.a3")]
    run = make_runner(wg, n_slots=4, cap=2048, path=path)
    case = Case(run, reqs, {0: 0, 1: synth.mask_of([1])})
    res = case.step()
    assert run.v.attention_kernel() == TC
    case.check(wo, res, f"{path} split")
    run.close()


@pytest.mark.parametrize("path", PATHS)
def test_tc_ctas_cover_several_items(weights, path):
    """Eight chains of 6 rows with contexts 2500-4000: about three tiles per CTA, so CTAs move
    from one item to the next (Q double buffer, per-item partials) and items span CTAs."""
    wo, wg = weights
    ctx = [2500 + int(x) for x in synth.uniform_ints(8, 1501, SEED, "tc.many.ctx").tolist()]
    reqs = [chain(c, 5, f"tc.m{b}", domain=b % 2) for b, c in enumerate(ctx)]
    run = make_runner(wg, n_slots=8, cap=4096 + 16, path=path)
    case = Case(run, reqs, {0: 0, 1: synth.mask_of([2])})
    res = case.step()
    assert run.v.attention_kernel() == TC
    case.check(wo, res, f"{path} many")
    run.close()


def test_tc_matches_warp_kernel_and_is_deterministic(weights):
    """The same step with the tcgen05 kernel twice (bitwise equal: the partials merge in CTA
    order) and with the warp-level kernel (both within the oracle's tolerance, and close)."""
    wo, wg = weights
    reqs = [chain(700, 5, "tc.d0"), tree16(1500, "tc.d1"), chain(64, 3, "tc.d2")]
    out = {}
    for tc in (True, False):
        run = make_runner(wg, n_slots=3, cap=2048, path="hybrid", tc=tc)
        case = Case(run, reqs, {0: 0})
        res = case.step()
        assert run.v.attention_kernel() == (TC if tc else NARROW)
        case.check(wo, res, f"tc={tc}")
        out[tc] = res["logits"].cpu().numpy().copy()
        if tc:
            for l in range(ARCH.n_layers):  # undo the step's appends, then the same step again
                for b, r in enumerate(reqs):
                    run.kv[l][b, :, :, r.ctx_len:].fill_(float("nan"))
            res2 = case.step()
            np.testing.assert_array_equal(res2["logits"].cpu().numpy(), out[True])
        run.close()
    assert float(np.abs(out[True] - out[False]).max()) < 2e-2


def test_tc_not_used_for_larger_blocks_or_when_off(weights):
    """Blocks over 16 rows keep the warp-level kernel; TSS_ATTN_TC=0 turns the tcgen05 kernel off."""
    wo, wg = weights
    from paper_2609_26100_gb300.runner import TssRunner
    os.environ.update({"TSS_PATH": "persistent", "TSS_ATTN": "external"})
    try:
        run = TssRunner(ARCH, wg, n_slots=1, kv_cap=1024, max_batch=8, max_nodes=32)
    finally:
        os.environ.pop("TSS_PATH", None)
        os.environ.pop("TSS_ATTN", None)
    case = Case(run, [chain(500, 19, "tc.big")], {0: 0})
    res = case.step()
    assert run.v.attention_kernel() == NARROW
    case.check(wo, res, "20 rows")
    run.close()


def test_tc_bounded_wait_times_out_and_the_context_recovers(weights):
    """Failure injection without a GPU fault, in the tcgen05 attention kernel: a step whose first
    attention launch has CTA 0 issue no MMA (tss_inject_timeout) ends with TSS_ERR_TIMEOUT from
    that kernel's bounded waits (2 s), every CTA drains its copies and frees its tensor memory,
    and the next steps on the same context run normally and match the oracle."""
    wo, wg = weights
    reqs = [chain(1000, 5, "tc.to0"), chain(300, 3, "tc.to1")]
    run = make_runner(wg, n_slots=2, cap=1024, path="hybrid")
    case = Case(run, reqs, {0: 0})
    run.v.inject_timeout(1)
    depth = max(max(synth.depths_of(r.parents)) for r in reqs)
    res = run.alloc_results(len(reqs), sum(len(r.parents) for r in reqs), path_stride=max(64, depth + 1))
    run.verify(run.batch(reqs), res)
    st = run.sync_status()
    torch.cuda.synchronize()
    assert st == native.TSS_ERR_TIMEOUT
    assert run.v.attention_kernel() == TC
    assert run.sync_status() == native.TSS_OK  # reported once, then cleared
    for _ in range(2):
        for l in range(ARCH.n_layers):  # the failed step's appends are discarded
            for b, r in enumerate(reqs):
                run.kv[l][b, :, :, r.ctx_len:].fill_(float("nan"))
        res = case.step()
        case.check(wo, res, "after a timeout")
    run.close()
