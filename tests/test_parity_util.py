"""The test-side sampling checks (no GPU): the fp64 walk on a logit matrix reproduces the
oracle's speculative sampling on the same matrix, spec_valid accepts exactly the results a walk
can give, and check_sample calls a perturbed matrix "flagged" only when the perturbation moves a
decision."""
import numpy as np

from oracle import tss_oracle as O
from paper_2609_26100_gb300 import synth
from tests.parity_util import check_sample, spec_valid, spec_walk


def _case(seed, V=64, k=4):
    rng = np.random.default_rng(seed)
    logits = rng.normal(0, 2.0, (k + 1, V))
    q = rng.dirichlet(np.ones(V), size=k + 1)
    toks = [int(rng.integers(V))] + [int(rng.choice(V, p=q[i])) for i in range(1, k + 1)]
    u = synth.uniform01(2 * k + 1, seed, "pu").double().numpy()
    return logits, q, toks, u


def test_walk_equals_the_oracle_rule():
    near_cases = 0
    for seed in range(300):
        logits, q, toks, u = _case(seed)
        a, b, _, _ = O.spec_sample_accept(logits, toks, q, u, 1.0)
        wa, wb, near = spec_walk(logits, toks, q, u, 1.0)
        near_cases += near
        if not near:
            assert (wa, wb) == (a, b)
        assert spec_valid(logits, toks, q, u, 1.0, a, b)
    assert near_cases < 10


def test_valid_rejects_other_results():
    logits, q, toks, u = _case(7)
    a, b, _, _ = O.spec_sample_accept(logits, toks, q, u, 1.0)
    assert spec_valid(logits, toks, q, u, 1.0, a, b)
    assert not spec_valid(logits, toks, q, u, 1.0, a, (b + 1) % 64) or q[min(a + 1, 4)][(b + 1) % 64] < 0
    for other in range(5):
        if other != a:
            assert not spec_valid(logits, toks, q, u, 1.0, other, b)


def test_check_sample_counts_moved_decisions_as_flagged():
    kinds = {"exact": 0, "flagged": 0, "slack": 0}
    for seed in range(200):
        logits, q, toks, u = _case(seed)
        noisy = logits + np.random.default_rng(seed + 1000).normal(0, 0.02, logits.shape)
        wa, wb, near = spec_walk(noisy, toks, q, u, 1.0)
        kinds[check_sample(logits, noisy, toks, q, u, 1.0, wa, wb)] += 1
    assert kinds["exact"] > 150 and kinds["flagged"] + kinds["slack"] > 0
