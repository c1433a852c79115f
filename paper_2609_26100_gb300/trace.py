"""Summary of the persistent verify kernel's device timeline.

With TSS_TRACE=1 set at tss_create, each CTA of the persistent kernel records globaltimer
nanoseconds of its roles' first and last activity in every phase of the last step, which
tss_read_trace (Verifier.read_trace) returns as one flat array.  The layout, per CTA:
  [pi * 8 + 2 * role + {0: first, 1: last}]  for phase pi -- QKV, O, gate/up, down of active
      layer slot j at pi = 4j .. 4j + 3, the LM head at pi = 4 n_act -- and role 0 weight
      copies, 1 B operand, 2 MMA, 3 epilogue;
  [ATTN_BASE + 2j + {0, 1}]  the CTA's attention items of slot j (first entry, last exit);
  further diagnostic slots follow.  0 means no activity.

summarize() turns that into, per phase, each role's window over the grid (earliest first,
median first, latest last; microseconds from the step's first recorded event) and, per layer
slot, the attention window and the layer's span from its first QKV weight copy to the last
epilogue of its down projection.
"""
from __future__ import annotations

from typing import Dict, List, Optional

import numpy as np

ROLES = ("weights", "b_operand", "mma", "epilogue")
KINDS = ("qkv", "o", "gate_up", "down")
MAX_LAYERS = 64
PHASES = 4 * MAX_LAYERS + 1
ATTN_BASE = PHASES * 8


def phase_name(pi: int, n_act: int):
    """(kind, layer slot) of phase pi."""
    if pi < 4 * n_act:
        return KINDS[pi % 4], pi // 4
    return "lm_head", n_act


def _window(first: np.ndarray, last: np.ndarray, t0: int) -> Optional[Dict[str, float]]:
    f = first[first > 0]
    l = last[last > 0]
    if f.size == 0 or l.size == 0:
        return None
    return {"first_min": (int(f.min()) - t0) / 1e3, "first_median": (float(np.median(f)) - t0) / 1e3,
            "last_max": (int(l.max()) - t0) / 1e3, "ctas": int(f.size)}


def summarize(trace, n_ctas: int, n_act: int) -> Dict:
    """Per-phase role windows, per-slot attention windows and layer spans (microseconds)."""
    tr = np.asarray(trace, dtype=np.uint64).reshape(n_ctas, -1).astype(np.int64)
    if tr.shape[1] < ATTN_BASE + 2 * MAX_LAYERS:
        raise ValueError(f"trace has {tr.shape[1]} slots per CTA, fewer than the layout needs")
    if not 0 <= n_act <= MAX_LAYERS:
        raise ValueError("n_act must be in [0, 64]")
    used = tr[:, : ATTN_BASE + 2 * MAX_LAYERS]
    nz = used[used > 0]
    if nz.size == 0:
        return {"phases": [], "attention": [], "layers": [], "total_us": 0.0}
    t0 = int(nz.min())
    phases: List[Dict] = []
    for pi in range(4 * n_act + 1):
        kind, slot = phase_name(pi, n_act)
        rec = {"phase": kind, "slot": slot}
        for r, role in enumerate(ROLES):
            rec[role] = _window(tr[:, pi * 8 + 2 * r], tr[:, pi * 8 + 2 * r + 1], t0)
        phases.append(rec)
    attention = []
    for j in range(n_act):
        attention.append({"slot": j, "window": _window(tr[:, ATTN_BASE + 2 * j], tr[:, ATTN_BASE + 2 * j + 1], t0)})
    layers = []
    for j in range(n_act):
        qkv_w = phases[4 * j]["weights"]
        down_e = phases[4 * j + 3]["epilogue"]
        if qkv_w and down_e:
            layers.append({"slot": j, "start": qkv_w["first_min"], "end": down_e["last_max"],
                           "span_us": down_e["last_max"] - qkv_w["first_min"]})
    return {"phases": phases, "attention": attention, "layers": layers, "total_us": (int(nz.max()) - t0) / 1e3}
