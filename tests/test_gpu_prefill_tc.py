"""GPU parity of the compute-bound prefill (tokens-tiled tcgen05 GEMMs and causal tcgen05
attention, head_dim 128) against the oracle's prefill, on a small decoder with 128-dimensional
heads (3 layers, d 256, 2 heads x 128, MLP 688, vocab 2048): prompts on empty caches and appended
to existing contexts, a prompt longer than one 1024-token chunk, requests of different skip sets,
partial token and query tiles, and a verification step on top of the GPU-filled cache."""
import os

import numpy as np
import pytest
import torch

from oracle import tss_oracle as O
from paper_2609_26100_gb300 import native, synth
from tests.conftest import oracle_weights
from tests.parity_util import assert_logits, to_device_weights

pytestmark = pytest.mark.gpu

ARCH = synth.Arch(n_layers=3, d_model=256, n_heads=2, head_dim=128, d_mlp=688, vocab=2048)
SEED = synth.DEFAULT_SEED


@pytest.fixture(scope="module")
def weights():
    from paper_2609_26100_gb300 import build
    build.build()
    w = synth.make_weights(ARCH)
    return oracle_weights(w), to_device_weights(w)


def make_runner(wg, n_slots, cap, prefill="tc"):
    from paper_2609_26100_gb300.runner import TssRunner
    env = {"TSS_PREFILL": "tc" if prefill == "tc" else "steps"}
    os.environ.update(env)
    try:
        return TssRunner(ARCH, wg, n_slots=n_slots, kv_cap=cap, max_batch=8, max_nodes=16)
    finally:
        for k in env:
            os.environ.pop(k, None)


def upload(run, kv, slot):
    for l, layer in enumerate(kv):
        if layer is not None:
            run.write_kv(l, slot, torch.from_numpy(layer[0]), torch.from_numpy(layer[1]))


@pytest.mark.parametrize("prefill", ["tc", "steps"])
def test_prefill_matches_oracle(weights, prefill):
    """Three requests: 300 tokens on an empty cache (skip {1}), 100 tokens after a 200-token
    context (dense), 1100 tokens on an empty cache (two chunks, skip {1}).  Every K/V row the
    oracle's prefill gives matches, skipped layers and rows past the prompt stay untouched, and a
    verification step on request 0's GPU-filled cache gives the oracle's logits."""
    wo, wg = weights
    phi = {0: O.set_to_mask({1}), 1: 0}
    run = make_runner(wg, n_slots=3, cap=1152, prefill=prefill)
    run.set_phi(phi)
    sentinel = 7.0
    for t in run.kv:
        t.fill_(sentinel)
    doms = [0, 1, 0]
    full = [synth.uniform_ints(300, ARCH.vocab, SEED, "pft.a").tolist(),
            synth.uniform_ints(300, ARCH.vocab, SEED, "pft.b").tolist(),
            synth.uniform_ints(1100, ARCH.vocab, SEED, "pft.c").tolist()]
    have = [0, 200, 0]
    skips = [O.skip_set({d: O.mask_to_set(m) for d, m in phi.items()}, d) for d in doms]
    upload(run, O.prefill(wo, ARCH, skips[1], full[1][:have[1]]), 1)
    run.prefill([full[b][have[b]:] for b in range(3)], have, doms)
    assert run.sync_status() == native.TSS_OK
    torch.cuda.synchronize()
    refs = [O.prefill(wo, ARCH, skips[b], full[b]) for b in range(3)]
    for b in range(3):
        C = len(full[b])
        for l in range(ARCH.n_layers):
            region = run.kv[l][b]
            if l in skips[b]:
                assert bool((region == sentinel).all()), f"request {b} skipped layer {l} was touched"
                continue
            gk = region[0, :, :C].float().cpu().numpy()
            gv = region[1, :, :C].float().cpu().numpy()
            np.testing.assert_allclose(gk, refs[b][l][0], atol=5e-2, rtol=3e-2, err_msg=f"K request {b} layer {l}")
            np.testing.assert_allclose(gv, refs[b][l][1], atol=5e-2, rtol=3e-2, err_msg=f"V request {b} layer {l}")
            assert float(np.abs(gk - refs[b][l][0]).mean()) < 2e-3
            assert bool((region[:, :, C:] == sentinel).all())
    # a verification step on the GPU-filled cache of request 0
    C = len(full[0])
    parents = synth.chain_parents(4)
    toks = synth.draft_tokens(parents, ARCH.vocab, SEED, "pft.tok")
    res = run.alloc_results(1, len(parents))
    run.verify(run.batch([synth.Request(C, parents, toks, doms[0])]), res)
    assert run.sync_status() == native.TSS_OK
    torch.cuda.synchronize()
    ref, _ = O.verify_request(wo, ARCH, skips[0], toks, parents, C, refs[0])
    assert_logits(res["logits"].cpu().numpy(), ref, f"verify after GPU prefill ({prefill})")
    run.close()


def test_prefill_nan_tail_and_empty_prompt(weights):
    """Cache rows past the prompt holding NaN never reach the attention (the last key tile's V
    rows past the keys are zeroed), and an empty prompt changes nothing."""
    wo, wg = weights
    run = make_runner(wg, n_slots=2, cap=512)
    run.set_phi({0: 0})
    for t in run.kv:
        t.fill_(float("nan"))
    full = synth.uniform_ints(130, ARCH.vocab, SEED, "pft.n").tolist()
    run.prefill([full, []], [0, 0], [0, 0])
    assert run.sync_status() == native.TSS_OK
    torch.cuda.synchronize()
    ref = O.prefill(wo, ARCH, frozenset(), full)
    for l in range(ARCH.n_layers):
        gk = run.kv[l][0, 0, :, :130].float().cpu().numpy()
        gv = run.kv[l][0, 1, :, :130].float().cpu().numpy()
        np.testing.assert_allclose(gk, ref[l][0], atol=5e-2, rtol=3e-2)
        np.testing.assert_allclose(gv, ref[l][1], atol=5e-2, rtol=3e-2)
        assert bool(torch.isnan(run.kv[l][1]).all())  # slot 1: untouched
    run.close()


def test_prefill_host_checks(weights):
    """Host-detectable errors return before any launch: a prompt past the KV capacity, a slot out
    of range, and positions past the context's max_positions (the RoPE tables' rows)."""
    wo, wg = weights
    run = make_runner(wg, n_slots=1, cap=256)
    run.set_phi({0: 0})
    with pytest.raises(native.TssError) as err:
        run.prefill([list(range(100))], [200], [0])
    assert err.value.status == native.TSS_ERR_KV_CAPACITY
    with pytest.raises(native.TssError) as err:
        run.prefill([list(range(10))], [0], [0], slots=[3])
    assert err.value.status == native.TSS_ERR_INVALID_ARG
    run.close()
    v = native.Verifier(wg, ARCH, max_batch=8, max_rows=256, max_nodes=16, max_positions=64)
    H, D = ARCH.n_heads, ARCH.head_dim
    cache = [torch.zeros((1, 2, H, 256, D), dtype=torch.bfloat16, device="cuda") for _ in range(ARCH.n_layers)]
    kv = v.make_kv([t.data_ptr() for t in cache], 1, 256)
    toks = torch.zeros(100, dtype=torch.int32, device="cuda")
    with pytest.raises(native.TssError) as err:
        v.prefill([100], [0], [0], toks, kv)
    assert err.value.status == native.TSS_ERR_INVALID_ARG
    assert "max_positions" in str(err.value)
    v.close()


def test_prefill_bounded_wait_times_out_and_recovers(weights):
    """Failure injection without a GPU fault, in the prefill GEMM: tss_inject_timeout makes CTA 0
    of the call's first GEMM issue no MMA; the call ends with TSS_ERR_TIMEOUT from the bounded
    waits (2 s), and the next prefill on the same context matches the oracle."""
    wo, wg = weights
    run = make_runner(wg, n_slots=1, cap=512)
    run.set_phi({0: 0})
    full = synth.uniform_ints(200, ARCH.vocab, SEED, "pft.to").tolist()
    run.v.inject_timeout(1)
    run.prefill([full], [0], [0])
    assert run.sync_status() == native.TSS_ERR_TIMEOUT
    assert run.sync_status() == native.TSS_OK  # reported once, then cleared
    run.prefill([full], [0], [0])
    assert run.sync_status() == native.TSS_OK
    torch.cuda.synchronize()
    ref = O.prefill(wo, ARCH, frozenset(), full)
    for l in range(ARCH.n_layers):
        np.testing.assert_allclose(run.kv[l][0, 0, :, :200].float().cpu().numpy(), ref[l][0], atol=5e-2, rtol=3e-2)
        np.testing.assert_allclose(run.kv[l][0, 1, :, :200].float().cpu().numpy(), ref[l][1], atol=5e-2, rtol=3e-2)
    run.close()
