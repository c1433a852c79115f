"""Offline search for a domain's skip configuration: the acceptance- and metric-aware breadth
search of Sec. "Acceptance- and Metric-Aware Breadth-First Search" (Algorithm 1), with the
verification cost C_d(S) taken from this library.

The search (Sec. "Problem Formulation"): among skip sets S of a target with L blocks, find the one
of lowest verification cost C_d(S) whose mean acceptance A_d(S) and task metric M_d(S) stay within
eps_A and eps_M of the dense verifier's (A_d^0, M_d^0).  Algorithm 1 in outline:

  1. evaluate the dense verifier (S = {}) for A_d^0, M_d^0, C_d^0;
  2. candidate pool L_d: every single layer l whose skip {l} keeps acceptance within tau_A of the
     dense value OR the metric within tau_M (a permissive "or", so that a layer useful for only
     one of the two survives);
  3. for depth k = 1..K, every k-subset of L_d is evaluated; the feasible ones (acceptance within
     eps_A AND metric within eps_M of the dense values) join F_d and the record set P_d; the
     search stops at the first depth with no feasible set;
  4. P_d loses its dominated records, and S_d* is the feasible set (the dense one included) of
     lowest cost.

Readings of points the paper leaves open (also in the repository's design notes):
  * layers are 0-based, as everywhere in this library;
  * each set is evaluated once (the single-layer sets of step 2 are reused at depth 1);
  * "dominated" compares acceptance and metric, as the section words it (a record is dropped when
    another has both at least as high and one higher); pareto_cost=True also compares the cost;
  * ties of the lowest cost go to the higher acceptance, then the higher metric, then the smaller
    set, then the lexicographically first: with a byte-count cost every set of one size costs the
    same;
  * the hyper-parameter table's "beam width" and "barriers" have no step in Algorithm 1 and are
    not used.

The objectives need calibration data and draft models that this repository does not have: A_d
and M_d come from a caller's evaluate(S), e.g. SyntheticObjective, a seeded stand-in with
per-layer effects and interactions between neighbouring layers.  C_d comes from the library:
bytes_cost (tss_estimate_step_bytes, host arithmetic; on this memory-bound path the step time is
proportional to it) or latency_cost (tss_verify timed with CUDA events on the GPU).
"""
from __future__ import annotations

import argparse
import itertools
import json
from dataclasses import dataclass, field
from typing import Callable, Dict, List, Optional, Sequence, Tuple

import numpy as np

SkipSet = Tuple[int, ...]


@dataclass(frozen=True)
class Evaluation:
    accept: float  # A_d(S): mean accepted draft tokens per verification step
    metric: float  # M_d(S): downstream task metric (higher is better)
    cost: float    # C_d(S): verification cost (lower is better)


@dataclass
class SearchResult:
    best: SkipSet                      # S_d*
    best_eval: Evaluation
    baseline: Evaluation               # (A_d^0, M_d^0, C_d^0)
    candidates: SkipSet                # L_d
    feasible: Dict[int, List[SkipSet]]  # F_d^(k) per depth k; depth 0 is the dense set
    pareto: List[Tuple[SkipSet, Evaluation]]  # P_d without dominated records
    evaluations: int                   # distinct sets evaluated
    depth: int                         # last depth evaluated
    log: List[Tuple[SkipSet, Evaluation]] = field(default_factory=list)  # every evaluation, in order


def dominates(x: Evaluation, y: Evaluation, with_cost: bool = False) -> bool:
    """x dominates y: at least as good in every compared objective, better in one."""
    ge = x.accept >= y.accept and x.metric >= y.metric and (not with_cost or x.cost <= y.cost)
    gt = x.accept > y.accept or x.metric > y.metric or (with_cost and x.cost < y.cost)
    return ge and gt


def breadth_search(n_layers: int, evaluate: Callable[[SkipSet], Evaluation], K: int, eps_a: float, eps_m: float,
                   tau_a: float, tau_m: float, layers: Optional[Sequence[int]] = None,
                   pareto_cost: bool = False) -> SearchResult:
    """Algorithm 1 over the layers `layers` (default: all n_layers, 0-based) up to depth K."""
    if K < 0:
        raise ValueError("K must be >= 0")
    pool_layers = list(range(n_layers)) if layers is None else sorted(set(int(l) for l in layers))
    if any(not 0 <= l < n_layers for l in pool_layers):
        raise ValueError("layers must lie in [0, n_layers)")
    seen: Dict[SkipSet, Evaluation] = {}
    log: List[Tuple[SkipSet, Evaluation]] = []

    def ev(s) -> Evaluation:
        key = tuple(sorted(s))
        if key not in seen:
            seen[key] = evaluate(key)
            log.append((key, seen[key]))
        return seen[key]

    base = ev(())
    # step 2: the permissive candidate pool ("or")
    candidates = tuple(l for l in pool_layers
                       if ev((l,)).accept >= base.accept - tau_a or ev((l,)).metric >= base.metric - tau_m)
    # step 3: depth by depth, the strict feasibility test ("and")
    feasible: Dict[int, List[SkipSet]] = {0: [()]}
    records: List[Tuple[SkipSet, Evaluation]] = [((), base)]
    depth = 0
    for k in range(1, K + 1):
        depth = k
        level = []
        for s in itertools.combinations(candidates, k):
            e = ev(s)
            if e.accept >= base.accept - eps_a and e.metric >= base.metric - eps_m:
                level.append(s)
                records.append((s, e))
        if not level:
            break
        feasible[k] = level
    # step 4: non-dominated records and the cheapest feasible set
    pareto = [(s, e) for s, e in records if not any(dominates(f, e, pareto_cost) for _, f in records)]
    every = [s for k in sorted(feasible) for s in feasible[k]]
    best = min(every, key=lambda s: (seen[s].cost, -seen[s].accept, -seen[s].metric, len(s), s))
    return SearchResult(best, seen[best], base, candidates, feasible, pareto, len(seen), depth, log)


# ----------------------------------------------------------------------------------------------
# Objectives and costs
# ----------------------------------------------------------------------------------------------
class SyntheticObjective:
    """Seeded stand-in for A_d(S) and M_d(S) (calibration data and draft models are not available):
    each skipped layer shifts acceptance by a_l and the metric by m_l (normal draws, a few layers
    helping, most hurting; later layers matter less), skipping two neighbouring layers costs
    extra (the effects are not additive), and the loss grows with the square of the number of
    skipped layers."""

    def __init__(self, n_layers: int, seed: int = 42, accept0: float = 3.0, metric0: float = 0.5):
        rng = np.random.default_rng(seed)
        depth = np.linspace(1.0, 0.3, n_layers)
        self.n_layers = n_layers
        self.accept0, self.metric0 = accept0, metric0
        self.a = rng.normal(-0.06, 0.12, n_layers) * depth
        self.m = rng.normal(-0.012, 0.02, n_layers) * depth
        self.pair_a = -0.08
        self.pair_m = -0.015

    def __call__(self, s: SkipSet) -> Tuple[float, float]:
        s = sorted(s)
        adj = sum(1 for x, y in zip(s, s[1:]) if y == x + 1)
        n = len(s)
        acc = self.accept0 + float(sum(self.a[l] for l in s)) + self.pair_a * adj - 0.01 * n * n
        met = self.metric0 + float(sum(self.m[l] for l in s)) + self.pair_m * adj - 0.002 * n * n
        return acc, met


def bytes_cost(arch, requests) -> Callable[[SkipSet], float]:
    """C_d(S) as the HBM bytes of one verification step of `requests` (synth.Request list) when
    every request skips S: tss_estimate_step_bytes, host arithmetic."""
    from . import native
    ctx = [r.ctx_len for r in requests]
    nodes = [len(r.parents) for r in requests]

    def cost(s: SkipSet) -> float:
        m = 0
        for l in s:
            m |= 1 << l
        return float(native.estimate_step_bytes(arch, [m] * len(requests), ctx, nodes)["total"])

    return cost


def latency_cost(runner, requests, steps: int = 10, warmup: int = 3, domain: int = 0) -> Callable[[SkipSet], float]:
    """C_d(S) as the measured time (microseconds, mean of `steps` CUDA-event-timed tss_verify
    calls) of one verification step of `requests` with every request's domain mapped to S."""
    import torch
    from . import synth

    reqs = [synth.Request(r.ctx_len, r.parents, r.tokens, domain) for r in requests]
    res = runner.alloc_results(len(reqs), sum(len(r.parents) for r in reqs), logits=False)
    batch = runner.batch(reqs)
    stream = torch.cuda.current_stream()

    def cost(s: SkipSet) -> float:
        m = 0
        for l in s:
            m |= 1 << l
        runner.set_phi({domain: m})
        for _ in range(warmup):
            runner.verify(batch, res)
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        for _ in range(steps):
            runner.verify(batch, res)
        e1.record(stream)
        torch.cuda.synchronize()
        return e0.elapsed_time(e1) / steps * 1e3

    return cost


def combine(objective: Callable[[SkipSet], Tuple[float, float]], cost: Callable[[SkipSet], float]):
    return lambda s: Evaluation(*objective(s), cost(s))


def to_phi_record(result: SearchResult, domain: int, n_layers: int, name: str = "") -> dict:
    """The domain's record G_d = (S_d, A_d, M_d, R_d) in the configuration-file format."""
    return {"id": domain, "name": name, "skip": list(result.best), "accept_len": result.best_eval.accept,
            "metric": result.best_eval.metric, "sparsity": len(result.best) / float(n_layers)}


def main(argv=None):
    p = argparse.ArgumentParser(description="Algorithm 1 over a synthetic objective with the library's cost")
    p.add_argument("--workload", default="7b_chain", choices=["7b_chain", "7b_tree", "tiny"])
    p.add_argument("--cost", default="bytes", choices=["bytes", "latency"])
    p.add_argument("--K", type=int, default=4)
    p.add_argument("--eps-accept", type=float, default=0.15)
    p.add_argument("--eps-metric", type=float, default=0.025)
    p.add_argument("--tau-accept", type=float, default=0.15)
    p.add_argument("--tau-metric", type=float, default=0.025)
    p.add_argument("--seed", type=int, default=42)
    p.add_argument("--domain", type=int, default=0)
    p.add_argument("--out", default=None, help="write the domain's record to this configuration file")
    args = p.parse_args(argv)
    from . import synth
    w = {"7b_chain": synth.workload_7b_chain, "7b_tree": synth.workload_7b_tree,
         "tiny": synth.workload_tiny}[args.workload]()
    a = w.arch
    if args.cost == "bytes":
        cost = bytes_cost(a, w.requests)
    else:
        from .runner import TssRunner
        cost = latency_cost(TssRunner.for_workload(synth.workload_7b_chain(mask_layers=()) if args.workload == "7b_chain"
                                                   else w), w.requests)
    res = breadth_search(a.n_layers, combine(SyntheticObjective(a.n_layers, args.seed), cost), args.K,
                         args.eps_accept, args.eps_metric, args.tau_accept, args.tau_metric)
    rec = to_phi_record(res, args.domain, a.n_layers, f"synthetic seed {args.seed}")
    out = {"best": list(res.best), "best_eval": vars(res.best_eval), "baseline": vars(res.baseline),
           "candidates": list(res.candidates), "feasible_per_depth": {k: len(v) for k, v in res.feasible.items()},
           "depth": res.depth, "evaluations": res.evaluations,
           "pareto": [[list(s), vars(e)] for s, e in res.pareto], "record": rec}
    if args.out:
        with open(args.out, "w") as f:
            json.dump({"n_layers": a.n_layers, "domains": [rec]}, f, indent=1)
    print(json.dumps(out))


if __name__ == "__main__":
    main()
