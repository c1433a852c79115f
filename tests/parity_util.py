"""Helpers shared by the GPU parity tests: tolerance checks, lockstep KV handling, near-tie
validity checks.  The expected values always come from the CPU oracle."""
import numpy as np
import torch

from oracle import tss_oracle as O

LOGIT_MAX_ABS = 5e-2  # parity bar on logits (bf16 weights, fp32 accumulate)
LOGIT_REL_L2 = 1e-2


def logits_close(gpu: np.ndarray, ref: np.ndarray):
    err = np.abs(gpu.astype(np.float64) - ref.astype(np.float64))
    rel = float(np.linalg.norm(gpu.astype(np.float64) - ref) / max(np.linalg.norm(ref), 1e-30))
    return float(err.max()), rel


def assert_logits(gpu, ref, what=""):
    mx, rel = logits_close(gpu, ref)
    print(f"[parity] {what}: logits max-abs {mx:.3e}, rel-L2 {rel:.3e}")
    assert mx <= LOGIT_MAX_ABS and rel <= LOGIT_REL_L2, f"{what}: logits max-abs {mx:.3e}, rel-L2 {rel:.3e}"
    return mx, rel


def to_device_weights(w, device="cuda"):
    return {
        "embed": w["embed"].to(device), "lm_head": w["lm_head"].to(device), "final_norm": w["final_norm"].to(device),
        "layers": [None if lw is None else {k: v.to(device) for k, v in lw.items()} for lw in w["layers"]],
    }


def kv_to_torch(kv_layer):
    """oracle (K [H, C, D], V) float32 holding bf16 values -> two bf16 torch tensors."""
    k, v = kv_layer
    return torch.from_numpy(np.ascontiguousarray(k)).to(torch.bfloat16), torch.from_numpy(np.ascontiguousarray(v)).to(torch.bfloat16)


def greedy_valid(logits: np.ndarray, tokens, parents, path, bonus, band: float = 2 * O.GREEDY_MARGIN) -> bool:
    """A greedy walk that differs from the oracle's at a near-tie is still valid if every choice it
    made is within ``band`` of the oracle row maximum and each step follows a real child."""
    ch = O.children_of(parents)
    for a, b in zip(path[:-1], path[1:]):
        if b not in ch[a]:
            return False
        if logits[a][tokens[b]] < logits[a].max() - band:
            return False
    last = path[-1]
    return logits[last][bonus] >= logits[last].max() - band


def gpu_path(res, b, a):
    return [int(x) for x in res["path"][b][: a + 1].tolist()]


# ----------------------------------------------------------------------------------------------
# Speculative sampling: exact on every decision the measured logit error cannot move
# ----------------------------------------------------------------------------------------------
SAMPLE_FP32_SLACK = 1e-5  # relative (accept tests) / absolute normalised mass (draws): the GPU's fp32 sums


def _softmax64(row, temperature):
    z = np.asarray(row, dtype=np.float64) / float(temperature)
    z = z - z.max()
    e = np.exp(z)
    return e / e.sum()


def _draw64(w, u, slack):
    c = np.cumsum(np.asarray(w, dtype=np.float64))
    cn = c / c[-1]
    v = min(int(np.searchsorted(cn, u, side="right")), len(c) - 1)
    lo = cn[v - 1] if v > 0 else 0.0
    return v, (u - lo) <= slack or (cn[v] - u) <= slack, lo, cn[v]


def spec_walk(rows, tokens, q, u, temperature, slack=SAMPLE_FP32_SLACK):
    """The speculative-sampling walk evaluated in fp64 on the given logit rows (the rule the oracle
    states: accept draft i iff u[i-1] q_i(x_i) < p_{i-1}(x_i); at the first rejection draw from
    norm(max(0, p_{i-1} - q_i)) with u[k+i-1]; else from p_k with u[2k]).  Returns (a, bonus, near):
    near = some decision lies within `slack` of its threshold, where fp32 arithmetic may go either
    way.  Test-side arithmetic on measured rows, used to tell which decisions the measured logit
    error moves; the expected values come from the oracle."""
    k = len(tokens) - 1
    near = False
    for i in range(1, k + 1):
        p = _softmax64(rows[i - 1], temperature)
        x = int(tokens[i])
        lhs, rhs = float(u[i - 1]) * float(q[i][x]), float(p[x])
        near = near or abs(lhs - rhs) <= slack * rhs
        if lhs < rhs:
            continue
        v, nb, _, _ = _draw64(np.maximum(p - np.asarray(q[i], dtype=np.float64), 0.0), float(u[k + i - 1]), slack)
        return i - 1, v, near or nb
    v, nb, _, _ = _draw64(_softmax64(rows[k], temperature), float(u[2 * k]), slack)
    return k, v, near or nb


def spec_valid(rows, tokens, q, u, temperature, a, bonus, slack=SAMPLE_FP32_SLACK) -> bool:
    """(a, bonus) is what the walk on `rows` gives once each decision within `slack` of its
    threshold may go either way."""
    k = len(tokens) - 1
    if not 0 <= a <= k:
        return False
    for i in range(1, a + 2):
        if i > k:
            break
        p = _softmax64(rows[i - 1], temperature)
        x = int(tokens[i])
        lhs, rhs = float(u[i - 1]) * float(q[i][x]), float(p[x])
        if i <= a and not lhs < rhs * (1 + slack):
            return False  # accepted a draft the rows reject
        if i == a + 1 and not lhs >= rhs * (1 - slack):
            return False  # rejected a draft the rows accept
    if a < k:
        w = np.maximum(_softmax64(rows[a], temperature) - np.asarray(q[a + 1], dtype=np.float64), 0.0)
        uu = float(u[k + a])
    else:
        w = _softmax64(rows[k], temperature)
        uu = float(u[2 * k])
    if not (0 <= bonus < len(w)) or w[bonus] <= 0.0:
        return False
    c = np.cumsum(w) / w.sum()
    lo = c[bonus - 1] if bonus > 0 else 0.0
    return lo - slack <= uu <= c[bonus] + slack


def check_sample(ref_rows, gpu_rows, tokens, q, u, temperature, ga, gb, what=""):
    """One request's speculative-sampling outcome against the oracle.  Returns "exact" (GPU equals
    the oracle), "flagged" (the GPU's own logits, within the logit tolerance of the oracle's, put a
    uniform on the other side of a threshold: the GPU must then equal the walk on its logits) or
    "slack" (a decision within fp32 rounding of its threshold on the GPU's logits: the GPU result
    must be a valid walk).  Never passes a result that is wrong for both rows."""
    oa, ob, _, _ = O.spec_sample_accept(ref_rows, tokens, q, u, temperature)
    wa, wb, near = spec_walk(gpu_rows, tokens, q, u, temperature)
    if near:
        assert spec_valid(gpu_rows, tokens, q, u, temperature, ga, gb), f"{what}: ({ga}, {gb}) invalid"
        return "exact" if (ga, gb) == (oa, ob) else "slack"
    assert (ga, gb) == (wa, wb), f"{what}: GPU ({ga}, {gb}) != walk on its own logits ({wa}, {wb})"
    return "exact" if (wa, wb) == (oa, ob) else "flagged"
