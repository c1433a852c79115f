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
