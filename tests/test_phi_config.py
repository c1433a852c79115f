"""The configuration file of the domain map Phi (host logic, no GPU): records round-trip, the
paper's Table 1 skip sets load with their printed sparsity, and malformed records are rejected
with the record at fault."""
import json
import os

import pytest

from paper_2609_26100_gb300 import phi_config as PC

GOLDEN = os.path.join(os.path.dirname(__file__), "golden", "table1_skip_sets.txt")


def _table1():
    rows = {}
    with open(GOLDEN) as f:
        for ln in f:
            if ln.strip() and not ln.startswith("#"):
                L, name, pct, layers = ln.split()
                rows.setdefault(int(L), []).append((name, float(pct), [int(x) for x in layers.split(",")]))
    return rows


def test_table1_sets_round_trip_with_their_printed_sparsity(tmp_path):
    for L, recs in _table1().items():
        cfgs = [PC.DomainConfig(i, tuple(sorted(s)), name) for i, (name, _, s) in enumerate(recs)]
        path = tmp_path / f"phi{L}.json"
        PC.save(str(path), L, cfgs)
        back = PC.load(str(path), L)
        assert [back[i] for i in range(len(cfgs))] == cfgs
        for i, (_, pct, s) in enumerate(recs):
            assert round(100 * back[i].sparsity(L), 1) == pct
            assert PC.masks(back)[i] == sum(1 << l for l in s)


def test_calibration_values_are_carried():
    c = PC.DomainConfig(3, (3, 25, 30), "translation", accept_len=4.53, metric=0.31)
    back = PC.parse(PC.dumps(32, [c]), 32)
    assert back[3] == c and back[3].mask() == (1 << 3) | (1 << 25) | (1 << 30)


def _doc(**rec):
    base = {"id": 0, "skip": [1, 2]}
    base.update(rec)
    return json.dumps({"n_layers": 32, "domains": [base]})


@pytest.mark.parametrize("text, why", [
    (_doc(skip=[1, 32]), "outside"),
    (_doc(skip=[-1]), "outside"),
    (_doc(skip=[4, 4]), "twice"),
    (_doc(id=-2), "non-negative"),
    (_doc(skip="1,2"), "list"),
    (_doc(sparsity=0.125), "sparsity"),
    (json.dumps({"n_layers": 65, "domains": []}), "n_layers"),
    (json.dumps({"n_layers": 32}), "keys"),
    (json.dumps({"n_layers": 32, "domains": [{"id": 1, "skip": []}, {"id": 1, "skip": [2]}]}), "twice"),
    ("{not json", "JSON"),
])
def test_malformed_records_are_rejected(text, why):
    with pytest.raises(ValueError, match=why):
        PC.parse(text)


def test_layer_count_must_match_the_model():
    with pytest.raises(ValueError, match="40 layers"):
        PC.parse(json.dumps({"n_layers": 40, "domains": []}), 32)
    assert PC.parse(_doc(sparsity=2 / 32), 32)[0].skip == (1, 2)


def test_runner_load_phi_sets_each_domain(tmp_path):
    """TssRunner.load_phi hands every record's bitmask to tss_set_skip_config (the verifier is
    replaced by a recorder, so no GPU is needed)."""
    from paper_2609_26100_gb300 import synth
    from paper_2609_26100_gb300.runner import TssRunner

    class Recorder:
        def __init__(self):
            self.calls = []

        def set_skip_config(self, domain, mask):
            self.calls.append((domain, mask))

    run = object.__new__(TssRunner)
    run.arch, run.v = synth.TINY, Recorder()
    path = tmp_path / "phi.json"
    PC.save(str(path), synth.TINY.n_layers, [PC.DomainConfig(5, (2,)), PC.DomainConfig(1, (0, 3))])
    assert run.load_phi(str(path)) == {1: 0b1001, 5: 0b100}
    assert sorted(run.v.calls) == [(1, 0b1001), (5, 0b100)]
    PC.save(str(path), 32, [PC.DomainConfig(0, (31,))])
    with pytest.raises(ValueError, match="32 layers"):
        run.load_phi(str(path))
