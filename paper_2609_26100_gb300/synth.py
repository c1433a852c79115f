"""Seeded synthetic inputs for the TSS verification path.

This module holds no part of the method's arithmetic.  It draws the *inputs* of a verify step
(random-init weights, token ids, draft trees, draft distributions, KV-cache contents and
per-domain skip sets) from a seed, and it is the one module that both sides of a parity test use:
the tests pass its values to the CPU oracle and, through the C ABI, to the CUDA library, and
``bench.py`` uses it to build the timed workload.

Every generator is a pure function of (seed, tag, element index) built from 32-bit integer
hashing carried in int64 torch arithmetic (every product stays below 2**63), followed by exact
integer-to-float conversion, one IEEE fp32 multiply (and add) and a round-to-nearest-even cast to
bf16.  The values are therefore identical whether a tensor is generated on the CPU or on a GPU.

Distributions (stand-ins for the paper's models and Spec-Bench inputs, whose checkpoints and
items are not used):

* linear and embedding weights: approximately N(0, 0.02^2), drawn as an Irwin-Hall sum of four
  uniform bytes (mean 510, variance 21845) scaled to the target standard deviation;
* RMSNorm gains: 1 + 0.1 * (the same unit-variance variate), so a kernel that ignores the gains
  cannot match;
* token ids: uniform over the vocabulary;
* synthetic KV rows: (byte - 128) / 128, exactly representable in bf16, uniform in [-1, 1);
* draft distributions q: softmax of unit-variance logits (the draft side is an input here).
"""
from __future__ import annotations

import dataclasses
import itertools
import math
import zlib
from typing import Dict, List, Optional, Sequence

import torch

_M32 = 0xFFFFFFFF
_MUL1 = 0x7FEB352D  # odd multipliers below 2**31, so (x < 2**32) * mul < 2**63
_MUL2 = 0x31848BAB
_CHUNK = 1 << 24
# Irwin-Hall(4) over bytes: mean 4 * 127.5, variance 4 * (256**2 - 1) / 12.
_IH_MEAN = 510
_IH_STD = math.sqrt(4 * (256 * 256 - 1) / 12.0)
# Positions per (layer, request, kind, head) in the synthetic-KV index space.
KV_POSITION_SPACE = 1 << 20


def _mix_int(x: int) -> int:
    x &= _M32
    x ^= x >> 16
    x = (x * _MUL1) & _M32
    x ^= x >> 15
    x = (x * _MUL2) & _M32
    x ^= x >> 16
    return x


def _mix(x: torch.Tensor) -> torch.Tensor:
    x = x ^ (x >> 16)
    x = (x * _MUL1) & _M32
    x = x ^ (x >> 15)
    x = (x * _MUL2) & _M32
    x = x ^ (x >> 16)
    return x


def _keys(seed: int, tag: str):
    t = zlib.crc32(tag.encode("utf-8")) & _M32
    k1 = _mix_int(_mix_int(seed & _M32) ^ t)
    k2 = _mix_int(k1 ^ 0x5BD1E995 ^ ((seed >> 32) & _M32))
    return k1, k2


def hash32(index: torch.Tensor, seed: int, tag: str) -> torch.Tensor:
    """32-bit hash (as int64 in [0, 2**32)) of each int64 element index under (seed, tag)."""
    k1, k2 = _keys(seed, tag)
    lo = index & _M32
    hi = index >> 32
    hw = _mix(hi ^ k2)
    return _mix(((_mix(lo ^ k1) + hw) & _M32) ^ k2)


def _gen(n: int, seed: int, tag: str, device, fn, out_dtype, start: int = 0) -> torch.Tensor:
    out = torch.empty(n, dtype=out_dtype, device=device)
    for a in range(0, n, _CHUNK):
        b = min(n, a + _CHUNK)
        idx = torch.arange(start + a, start + b, dtype=torch.int64, device=device)
        out[a:b] = fn(hash32(idx, seed, tag))
    return out


def _unit_normal(h: torch.Tensor) -> torch.Tensor:
    s = (h & 255) + ((h >> 8) & 255) + ((h >> 16) & 255) + (h >> 24)
    return (s - _IH_MEAN).to(torch.float32)


def normal_bf16(shape, seed: int, tag: str, std: float, mean: float = 0.0, device="cpu") -> torch.Tensor:
    """bf16 tensor with approximately N(mean, std^2) entries (Irwin-Hall of four bytes)."""
    n = int(math.prod(shape))
    scale = torch.tensor(std / _IH_STD, dtype=torch.float32, device=device)
    shift = torch.tensor(mean, dtype=torch.float32, device=device)

    def fn(h):
        z = _unit_normal(h) * scale
        if mean != 0.0:
            z = z + shift
        return z.to(torch.bfloat16)

    return _gen(n, seed, tag, device, fn, torch.bfloat16).view(*shape)


def uniform_ints(n: int, high: int, seed: int, tag: str, device="cpu") -> torch.Tensor:
    """int64 tensor of n ids uniform over [0, high) (hash modulo high)."""
    return _gen(n, seed, tag, device, lambda h: h % high, torch.int64)


def uniform01(n: int, seed: int, tag: str, device="cpu") -> torch.Tensor:
    """float64 tensor of n uniforms in [0, 1) with 32-bit resolution."""
    return _gen(n, seed, tag, device, lambda h: h.to(torch.float64) / 4294967296.0, torch.float64)


# ----------------------------------------------------------------------------------------------
# Model shapes (App. "Models": Vicuna-7B / Llama-2-13B are LLaMA decoders; the tiny shape is the
# small parity configuration).
# ----------------------------------------------------------------------------------------------
@dataclasses.dataclass(frozen=True)
class Arch:
    n_layers: int
    d_model: int
    n_heads: int
    head_dim: int
    d_mlp: int
    vocab: int
    rms_eps: float = 1e-5
    rope_theta: float = 1e4

    @property
    def kv_bytes_per_token(self) -> int:
        return 2 * self.d_model * 2

    @property
    def layer_weight_bytes(self) -> int:
        d, f = self.d_model, self.d_mlp
        return 2 * (4 * d * d + 3 * d * f)


TINY = Arch(n_layers=4, d_model=256, n_heads=4, head_dim=64, d_mlp=688, vocab=2048)
LLAMA2_7B = Arch(n_layers=32, d_model=4096, n_heads=32, head_dim=128, d_mlp=11008, vocab=32000)
LLAMA2_13B = Arch(n_layers=40, d_model=5120, n_heads=40, head_dim=128, d_mlp=13824, vocab=32000)

DEFAULT_SEED = 42  # Table "Default hyperparameters": random seed 42

LAYER_KEYS = ("attn_norm", "wq", "wk", "wv", "wo", "mlp_norm", "w_gate", "w_up", "w_down")


def layer_shapes(arch: Arch) -> Dict[str, tuple]:
    d, f = arch.d_model, arch.d_mlp
    return {
        "attn_norm": (d,), "wq": (d, d), "wk": (d, d), "wv": (d, d), "wo": (d, d),
        "mlp_norm": (d,), "w_gate": (f, d), "w_up": (f, d), "w_down": (d, f),
    }


def make_layer(arch: Arch, layer: int, seed: int = DEFAULT_SEED, device="cpu") -> Dict[str, torch.Tensor]:
    out = {}
    for key, shape in layer_shapes(arch).items():
        tag = f"layer{layer}.{key}"
        if key.endswith("norm"):
            out[key] = normal_bf16(shape, seed, tag, std=0.1, mean=1.0, device=device)
        else:
            out[key] = normal_bf16(shape, seed, tag, std=0.02, device=device)
    return out


def make_weights(arch: Arch, seed: int = DEFAULT_SEED, device="cpu", layers: Optional[Sequence[int]] = None):
    """Random-init bf16 weights of a LLaMA decoder, row-major [out][in].

    ``layers`` restricts generation to those layer indices (others are None), which lets a test
    or a timing sample skip layers it never runs.
    """
    want = set(range(arch.n_layers)) if layers is None else set(layers)
    return {
        "embed": normal_bf16((arch.vocab, arch.d_model), seed, "embed", std=0.02, device=device),
        "lm_head": normal_bf16((arch.vocab, arch.d_model), seed, "lm_head", std=0.02, device=device),
        "final_norm": normal_bf16((arch.d_model,), seed, "final_norm", std=0.1, mean=1.0, device=device),
        "layers": [make_layer(arch, l, seed, device) if l in want else None for l in range(arch.n_layers)],
    }


# ----------------------------------------------------------------------------------------------
# Draft structures
# ----------------------------------------------------------------------------------------------
def chain_parents(k: int) -> List[int]:
    """Parent array of a chain draft: root (row 0) followed by k draft tokens."""
    return [-1] + list(range(k))


def eagle_tree(n_nodes: int = 60, branching: Sequence[int] = (4, 3, 2, 2, 1, 1)) -> List[int]:
    """Parent array (root first) of a static draft tree of n_nodes draft nodes.

    Nodes are rank tuples (r_1..r_t), r_j < branching[j-1], t <= len(branching); they are ordered
    by (sum of ranks, depth, lexicographic ranks) and the first n_nodes are kept.  A prefix of a
    tuple always sorts before it, so the kept set is closed under prefixes and the order is
    topological.
    """
    tuples = []
    for t in range(1, len(branching) + 1):
        tuples.extend(itertools.product(*[range(b) for b in branching[:t]]))
    tuples.sort(key=lambda r: (sum(r), len(r), r))
    kept = tuples[:n_nodes]
    index = {(): 0}
    parents = [-1]
    for i, r in enumerate(kept, start=1):
        index[r] = i
        parents.append(index[r[:-1]])
    return parents


def depths_of(parents: Sequence[int]) -> List[int]:
    d = []
    for i, p in enumerate(parents):
        d.append(0 if p < 0 else d[p] + 1)
    return d


def draft_tokens(parents: Sequence[int], vocab: int, seed: int, tag: str) -> List[int]:
    """Token ids for a draft block: row 0 (the root, last committed token) and every node,
    with siblings drawn without replacement so that no two children of a node share a token."""
    n = len(parents)
    raw = uniform_ints(4 * n + 64, vocab, seed, tag).tolist()
    src = iter(raw)
    toks = [0] * n
    used: Dict[int, set] = {}
    for i, p in enumerate(parents):
        taken = used.setdefault(p, set())
        t = next(src)
        while t in taken:
            t = next(src)
        taken.add(t)
        toks[i] = t
    return toks


def draft_probs_and_samples(n_rows: int, vocab: int, seed: int, tag: str):
    """Draft distributions q (softmax of unit-variance logits, float32 [n_rows][vocab]) and one
    token sampled from each row by inverse CDF with a hashed uniform."""
    z = normal_bf16((n_rows, vocab), seed, tag + ".logits", std=1.0).to(torch.float64)
    q = torch.softmax(z, dim=-1).to(torch.float32)
    u = uniform01(n_rows, seed, tag + ".u")
    c = torch.cumsum(q.to(torch.float64), dim=-1)
    idx = torch.searchsorted(c, (u * c[:, -1]).unsqueeze(1), right=True).squeeze(1)
    idx = torch.clamp(idx, max=vocab - 1)
    return q, [int(i) for i in idx.tolist()]


# ----------------------------------------------------------------------------------------------
# Skip sets and domains
# ----------------------------------------------------------------------------------------------
def mask_of(layers: Sequence[int]) -> int:
    m = 0
    for l in layers:
        m |= 1 << int(l)
    return m


def layers_of(mask: int) -> List[int]:
    return [l for l in range(64) if (mask >> l) & 1]


def seeded_subset(pool: Sequence[int], k: int, seed: int, tag: str) -> List[int]:
    """k distinct members of pool chosen by a seeded hash permutation, returned sorted."""
    keys = uniform_ints(len(pool), 1 << 30, seed, tag).tolist()
    order = sorted(range(len(pool)), key=lambda i: (keys[i], i))
    return sorted(pool[i] for i in order[:k])


def seeded_permutation(pool: Sequence[int], seed: int, tag: str) -> List[int]:
    keys = uniform_ints(len(pool), 1 << 30, seed, tag).tolist()
    order = sorted(range(len(pool)), key=lambda i: (keys[i], i))
    return [pool[i] for i in order]


# ----------------------------------------------------------------------------------------------
# Synthetic KV cache contents
# ----------------------------------------------------------------------------------------------
def kv_block(arch: Arch, layer: int, req: int, n_pos: int, seed: int, device="cpu", pos0: int = 0) -> torch.Tensor:
    """Synthetic bf16 K and V for positions [pos0, pos0 + n_pos) of one request in one layer,
    shaped [2][n_heads][n_pos][head_dim]; values (byte - 128) / 128.  Value at a position does
    not depend on the cache capacity or on n_pos."""
    H, D = arch.n_heads, arch.head_dim
    out = torch.empty((2, H, n_pos, D), dtype=torch.bfloat16, device=device)
    inv = torch.tensor(1.0 / 128.0, dtype=torch.float32, device=device)
    pos = torch.arange(pos0, pos0 + n_pos, dtype=torch.int64, device=device)
    dim = torch.arange(D, dtype=torch.int64, device=device)
    step = max(1, _CHUNK // max(1, D))
    for kind in range(2):
        for h in range(H):
            base = (((layer * 4096 + req) * 2 + kind) * H + h) * KV_POSITION_SPACE
            for a in range(0, n_pos, step):
                b = min(n_pos, a + step)
                idx = (base + pos[a:b]).unsqueeze(1) * D + dim.unsqueeze(0)
                hv = hash32(idx, seed, "kv")
                out[kind, h, a:b] = (((hv >> 24) - 128).to(torch.float32) * inv).to(torch.bfloat16)
    return out


# ----------------------------------------------------------------------------------------------
# Configurations (shapes and input recipes; the paper's Spec-Bench items are not used)
# ----------------------------------------------------------------------------------------------
@dataclasses.dataclass
class Request:
    ctx_len: int
    parents: List[int]
    tokens: List[int]
    domain: int
    draft_probs: Optional[torch.Tensor] = None  # [n_nodes][vocab] float32 (SAMPLE mode)


@dataclasses.dataclass
class Workload:
    name: str
    arch: Arch
    seed: int
    requests: List[Request]
    phi: Dict[int, int]  # domain id -> skip bitmask
    mode: str = "greedy"  # or "sample"
    temperature: float = 1.0
    kv_source: str = "synthetic"  # or "prefill" (oracle prefill of a random-id context)

    @property
    def n_rows(self) -> int:
        return sum(len(r.parents) for r in self.requests)

    def skip_mask(self, b: int) -> int:
        return self.phi.get(self.requests[b].domain, 0)

    def active_union(self) -> List[int]:
        L = self.arch.n_layers
        return [l for l in range(L) if any(not (self.skip_mask(b) >> l) & 1 for b in range(len(self.requests)))]


def config_chain(arch: Arch, name: str, batch: int, ctx: Sequence[int], k: int, phi: Dict[int, int],
                 domains: Sequence[int], seed: int = DEFAULT_SEED, mode: str = "greedy",
                 kv_source: str = "synthetic") -> Workload:
    reqs = []
    for b in range(batch):
        parents = chain_parents(k)
        if mode == "sample":
            q, samp = draft_probs_and_samples(len(parents), arch.vocab, seed, f"{name}.q{b}")
            root = uniform_ints(1, arch.vocab, seed, f"{name}.root{b}").item()
            toks = [int(root)] + samp[1:]
            reqs.append(Request(ctx[b], parents, toks, domains[b], q))
        else:
            toks = draft_tokens(parents, arch.vocab, seed, f"{name}.tok{b}")
            reqs.append(Request(ctx[b], parents, toks, domains[b]))
    return Workload(name, arch, seed, reqs, dict(phi), mode=mode, kv_source=kv_source)


def workload_tiny(mask_layers: Sequence[int] = (2,), seed: int = DEFAULT_SEED) -> Workload:
    """Tiny decoder, batch 1, 128-token context (oracle prefill), chain k=4, greedy."""
    return config_chain(TINY, "tiny", 1, [128], 4, {0: mask_of(mask_layers)}, [0], seed,
                        kv_source="prefill")


def workload_7b_chain(mask_layers: Sequence[int] = (20, 24, 27, 30), seed: int = DEFAULT_SEED,
                      ctx: int = 1024, k: int = 5) -> Workload:
    """7B shape, batch 1, context 1024, chain k=5, greedy; default skip set {20,24,27,30}."""
    return config_chain(LLAMA2_7B, "7b_chain", 1, [ctx], k, {0: mask_of(mask_layers)}, [0], seed)


def workload_7b_tree(seed: int = DEFAULT_SEED, ctx: int = 2048) -> Workload:
    """7B shape, 60-node draft tree, context 2048, 6 skipped layers drawn from 16..31."""
    arch = LLAMA2_7B
    parents = eagle_tree(60, (4, 3, 2, 2, 1, 1))
    toks = draft_tokens(parents, arch.vocab, seed, "7b_tree.tok")
    skip = seeded_subset(list(range(16, 32)), 6, seed, "7b_tree.skip")
    return Workload("7b_tree", arch, seed, [Request(ctx, parents, toks, 0)], {0: mask_of(skip)})


def workload_13b_mixed(seed: int = DEFAULT_SEED) -> Workload:
    """13B shape, batch 8, per-request context uniform in [512, 4096], 6 domains each skipping
    2..8 layers, chain k=5, speculative sampling at temperature 1."""
    arch = LLAMA2_13B
    phi = {}
    for d in range(6):
        n = 2 + int(uniform_ints(1, 7, seed, f"13b.nskip{d}").item())
        phi[d] = mask_of(seeded_subset(list(range(arch.n_layers)), n, seed, f"13b.skip{d}"))
    ctx = [512 + int(x) for x in uniform_ints(8, 4096 - 512 + 1, seed, "13b.ctx").tolist()]
    doms = [int(x) for x in uniform_ints(8, 6, seed, "13b.dom").tolist()]
    return config_chain(arch, "13b_mixed", 8, ctx, 5, phi, doms, seed, mode="sample")


def workload_7b_long(n_skip: int = 8, seed: int = DEFAULT_SEED, batch: int = 16, ctx: int = 16384,
                     k: int = 8) -> Workload:
    """7B shape, KV-bound: batch 16, context 16384, chain k=8.  Skip sets for the sweep are nested:
    the first n_skip layers of a seeded permutation of layers 1..31."""
    perm = seeded_permutation(list(range(1, LLAMA2_7B.n_layers)), seed, "7b_long.perm")
    skip = sorted(perm[:n_skip])
    return config_chain(LLAMA2_7B, "7b_long", batch, [ctx] * batch, k, {0: mask_of(skip)}, [0] * batch, seed)


def algorithmic_bytes(w: Workload) -> Dict[str, int]:
    """Bytes a verify step must move: weights of the union of active layers (once), the LM head,
    each request's active-layer KV context, and the new KV rows written."""
    a = w.arch
    union = w.active_union()
    weights = len(union) * a.layer_weight_bytes + a.vocab * a.d_model * 2
    kv_read = 0
    kv_write = 0
    for b, r in enumerate(w.requests):
        n_act = sum(1 for l in range(a.n_layers) if not (w.skip_mask(b) >> l) & 1)
        kv_read += n_act * r.ctx_len * a.kv_bytes_per_token
        kv_write += n_act * len(r.parents) * a.kv_bytes_per_token
    return {"weights": weights, "kv_read": kv_read, "kv_write": kv_write,
            "total": weights + kv_read + kv_write, "active_union": len(union)}
