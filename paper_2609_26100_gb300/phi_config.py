"""The domain-to-configuration map Phi kept as a small local file (Sec. "Domain-to-Configuration
Mapping"): after the offline search, each supported domain d has a record
G_d = (S_d, A_d(S_d), M_d(S_d), R_d) with R_d = |S_d| / L, and at run time the controller applies
S_d to the requests of domain d (Sec. "Domain-Aware Skip Controller").

File format (JSON, layer indices 0-based):

    {"n_layers": 32,
     "domains": [{"id": 0, "name": "translation", "skip": [3, 25, 30],
                  "accept_len": 4.53, "metric": 0.31, "sparsity": 0.09375}, ...]}

"skip" is S_d.  "accept_len" and "metric" are the calibrated A_d and M_d; the verifier does not
use them, so they are optional and carried as given.  "sparsity" is R_d; it is optional, and
when present it must equal |S_d| / L to within 5e-4.  load() checks every field and raises
ValueError with the record at fault.  masks() gives the bitmasks that tss_set_skip_config takes.
"""
from __future__ import annotations

import json
from dataclasses import dataclass
from typing import Dict, Iterable, Optional, Tuple

MAX_LAYERS = 64  # a skip set is a 64-bit mask in the C ABI


@dataclass(frozen=True)
class DomainConfig:
    domain: int
    skip: Tuple[int, ...]  # S_d, ascending
    name: str = ""
    accept_len: Optional[float] = None  # A_d(S_d)
    metric: Optional[float] = None      # M_d(S_d)

    def sparsity(self, n_layers: int) -> float:
        """R_d = |S_d| / L."""
        return len(self.skip) / float(n_layers)

    def mask(self) -> int:
        m = 0
        for l in self.skip:
            m |= 1 << l
        return m


def _check_layers(n_layers) -> int:
    if not isinstance(n_layers, int) or isinstance(n_layers, bool) or not 1 <= n_layers <= MAX_LAYERS:
        raise ValueError(f"n_layers must be an integer in [1, {MAX_LAYERS}], got {n_layers!r}")
    return n_layers


def _record(rec, n_layers: int, seen: set) -> DomainConfig:
    if not isinstance(rec, dict):
        raise ValueError(f"domain record must be an object, got {rec!r}")
    dom = rec.get("id")
    if not isinstance(dom, int) or isinstance(dom, bool) or dom < 0:
        raise ValueError(f"domain id must be a non-negative integer: {rec!r}")
    if dom in seen:
        raise ValueError(f"domain id {dom} appears twice")
    seen.add(dom)
    skip = rec.get("skip")
    if not isinstance(skip, list) or not all(isinstance(l, int) and not isinstance(l, bool) for l in skip):
        raise ValueError(f"domain {dom}: skip must be a list of layer indices")
    if len(set(skip)) != len(skip):
        raise ValueError(f"domain {dom}: skip lists a layer twice")
    bad = [l for l in skip if not 0 <= l < n_layers]
    if bad:
        raise ValueError(f"domain {dom}: layers {bad} outside [0, {n_layers})")
    cfg = DomainConfig(dom, tuple(sorted(skip)), str(rec.get("name", "")),
                       None if rec.get("accept_len") is None else float(rec["accept_len"]),
                       None if rec.get("metric") is None else float(rec["metric"]))
    if rec.get("sparsity") is not None and abs(float(rec["sparsity"]) - cfg.sparsity(n_layers)) > 5e-4:
        raise ValueError(f"domain {dom}: sparsity {rec['sparsity']} differs from |S|/L = "
                         f"{len(skip)}/{n_layers} = {cfg.sparsity(n_layers):.6f}")
    return cfg


def parse(text: str, n_layers: Optional[int] = None) -> Dict[int, DomainConfig]:
    """Records of a configuration file's text; n_layers, when given, must match the file's."""
    try:
        doc = json.loads(text)
    except json.JSONDecodeError as e:
        raise ValueError(f"not a JSON configuration file: {e}") from None
    if not isinstance(doc, dict) or "domains" not in doc:
        raise ValueError("configuration file needs the keys n_layers and domains")
    L = _check_layers(doc.get("n_layers"))
    if n_layers is not None and L != n_layers:
        raise ValueError(f"configuration is for {L} layers, the model has {n_layers}")
    if not isinstance(doc["domains"], list):
        raise ValueError("domains must be a list of records")
    seen: set = set()
    out = {}
    for rec in doc["domains"]:
        cfg = _record(rec, L, seen)
        out[cfg.domain] = cfg
    return out


def load(path: str, n_layers: Optional[int] = None) -> Dict[int, DomainConfig]:
    with open(path, encoding="utf-8") as f:
        return parse(f.read(), n_layers)


def dumps(n_layers: int, configs: Iterable[DomainConfig]) -> str:
    L = _check_layers(n_layers)
    recs = []
    for c in sorted(configs, key=lambda c: c.domain):
        r = {"id": c.domain, "name": c.name, "skip": list(c.skip), "sparsity": c.sparsity(L)}
        if c.accept_len is not None:
            r["accept_len"] = c.accept_len
        if c.metric is not None:
            r["metric"] = c.metric
        recs.append(r)
    text = json.dumps({"n_layers": L, "domains": recs}, indent=1)
    parse(text, L)  # what is written must load
    return text


def save(path: str, n_layers: int, configs: Iterable[DomainConfig]) -> None:
    text = dumps(n_layers, configs)
    with open(path, "w", encoding="utf-8") as f:
        f.write(text + "\n")


def masks(configs: Dict[int, DomainConfig]) -> Dict[int, int]:
    """domain id -> skip bitmask (bit l set = skip layer l), as tss_set_skip_config takes it."""
    return {d: c.mask() for d, c in configs.items()}
