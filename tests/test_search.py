"""Algorithm 1 (acceptance- and metric-aware breadth search) against brute force on small L (no
GPU): the candidate pool, the level-k sets, the feasibility test, the stop rule, the Pareto
pruning and the argmin, each recomputed here from its definition over every subset."""
import itertools
import json

import numpy as np
import pytest

from paper_2609_26100_gb300 import phi_config, search, synth
from paper_2609_26100_gb300.search import Evaluation


def _table(L, seed, cost_noise=True):
    """A random objective over every subset of L layers (a lookup table, not additive)."""
    rng = np.random.default_rng(seed)
    tab = {}
    for k in range(L + 1):
        for s in itertools.combinations(range(L), k):
            acc = 3.0 + rng.normal(-0.05 * k, 0.1)
            met = 0.5 + rng.normal(-0.01 * k, 0.02)
            cost = 100.0 - 10 * k + (rng.uniform(0, 1) if cost_noise else 0.0)
            tab[s] = Evaluation(acc, met, cost)
    return tab


def _brute(L, tab, K, ea, em, ta, tm, with_cost=False):
    base = tab[()]
    pool = tuple(l for l in range(L) if tab[(l,)].accept >= base.accept - ta or tab[(l,)].metric >= base.metric - tm)
    feas = {0: [()]}
    recs = [((), base)]
    depth = 0
    for k in range(1, K + 1):
        depth = k
        lv = [s for s in itertools.combinations(pool, k)
              if tab[s].accept >= base.accept - ea and tab[s].metric >= base.metric - em]
        recs += [(s, tab[s]) for s in lv]
        if not lv:
            break
        feas[k] = lv

    def dom(x, y):
        if with_cost:
            return (x.accept >= y.accept and x.metric >= y.metric and x.cost <= y.cost
                    and (x.accept > y.accept or x.metric > y.metric or x.cost < y.cost))
        return x.accept >= y.accept and x.metric >= y.metric and (x.accept > y.accept or x.metric > y.metric)

    pareto = [(s, e) for s, e in recs if not any(dom(f, e) for _, f in recs)]
    allf = [s for k in feas for s in feas[k]]
    lowest = min(tab[s].cost for s in allf)
    ties = [s for s in allf if tab[s].cost == lowest]
    return pool, feas, pareto, ties, depth


@pytest.mark.parametrize("seed", range(12))
@pytest.mark.parametrize("with_cost", [False, True])
def test_matches_brute_force(seed, with_cost):
    L, K = 8, 4
    tab = _table(L, seed)
    thr = dict(eps_a=0.12, eps_m=0.03, tau_a=0.08, tau_m=0.02)
    res = search.breadth_search(L, lambda s: tab[s], K, pareto_cost=with_cost, **thr)
    pool, feas, pareto, ties, depth = _brute(L, tab, K, thr["eps_a"], thr["eps_m"], thr["tau_a"], thr["tau_m"],
                                             with_cost)
    assert res.candidates == pool
    assert res.feasible == feas
    assert res.depth == depth
    assert sorted(res.pareto) == sorted(pareto)
    assert res.best in ties and len(ties) == 1  # costs carry noise: a unique argmin
    assert res.best_eval == tab[res.best] and res.baseline == tab[()]
    # evaluated: the dense set, every single layer, and the subsets of the pool up to the last depth
    expect = {()} | {(l,) for l in range(L)}
    for k in range(1, depth + 1):
        expect |= set(itertools.combinations(pool, k))
    assert res.evaluations == len(expect) and {s for s, _ in res.log} == expect


def test_or_pool_and_strict_feasibility():
    """A layer that keeps only the metric joins the pool (or), but a set that keeps only the metric
    is not feasible (and); a pair of feasible layers can be infeasible together."""
    base = Evaluation(3.0, 0.5, 100.0)
    tab = {(): base, (0,): Evaluation(2.0, 0.5, 90.0), (1,): Evaluation(3.0, 0.5, 90.0),
           (2,): Evaluation(3.0, 0.5, 90.0), (0, 1): Evaluation(3.0, 0.5, 80.0),
           (0, 2): Evaluation(3.0, 0.5, 80.0), (1, 2): Evaluation(2.5, 0.5, 80.0), (0, 1, 2): Evaluation(3, 0.5, 70.0)}
    res = search.breadth_search(3, lambda s: tab[s], 3, eps_a=0.1, eps_m=0.01, tau_a=0.1, tau_m=0.01)
    assert res.candidates == (0, 1, 2)  # layer 0 via the metric alone
    assert res.feasible[1] == [(1,), (2,)]  # {0} fails the acceptance bound
    assert res.feasible[2] == [(0, 1), (0, 2)]  # {1, 2} fails although both singles pass
    assert res.feasible[3] == [(0, 1, 2)]
    assert res.best == (0, 1, 2)


def test_stops_at_the_first_depth_without_a_feasible_set():
    calls = []

    def ev(s):
        calls.append(s)
        return Evaluation(3.0 - (0.5 if len(s) >= 2 else 0.0), 0.5, 100.0 - len(s))

    res = search.breadth_search(6, ev, 5, eps_a=0.1, eps_m=0.1, tau_a=0.1, tau_m=0.1)
    assert res.depth == 2 and 2 not in res.feasible
    assert max(len(s) for s in calls) == 2  # depth 3 is never evaluated
    assert len(res.best) == 1


def test_dense_is_the_answer_when_nothing_is_feasible():
    res = search.breadth_search(4, lambda s: Evaluation(3.0 - len(s), 0.5 - len(s), 10.0 - len(s)), 3, 0.1, 0.1, 0.1, 0.1)
    assert res.candidates == () and res.best == () and res.feasible == {0: [()]}


def test_byte_cost_ranks_by_active_layers_and_search_writes_a_config(tmp_path):
    """With the library's step-byte cost every skipped layer saves one layer's weights and KV, so
    the search picks the deepest feasible set; its record loads as a configuration file."""
    w = synth.workload_7b_chain()
    a = w.arch
    cost = search.bytes_cost(a, w.requests)
    assert cost(()) > cost((5,)) > cost((5, 9))
    assert cost((5,)) == cost((17,))
    obj = search.SyntheticObjective(a.n_layers, 42)
    res = search.breadth_search(a.n_layers, search.combine(obj, cost), 2, 0.15, 0.025, 0.15, 0.025)
    assert len(res.best) == max(res.feasible)
    rec = search.to_phi_record(res, 3, a.n_layers, "synthetic")
    path = tmp_path / "phi.json"
    path.write_text(json.dumps({"n_layers": a.n_layers, "domains": [rec]}))
    cfg = phi_config.load(str(path), a.n_layers)
    assert cfg[3].skip == res.best and abs(cfg[3].sparsity(a.n_layers) - len(res.best) / 32) < 1e-12
