"""Plain CPU oracle for TSS target-side verification (NumPy).

TEST INFRASTRUCTURE ONLY.  This module is the slow, obviously-correct reference that the CUDA
library is checked against.  Only tests/, __graft_entry__.smoke() and bench.py's cpu_baseline leg
may import it; the library and its binding never do, and nothing here imports them.

It follows the paper "TSS: Target-Side Sparsification for Speculative Decoding in
Domain-Specific Large Language Models":

* Sec. "Problem Formulation": a skip configuration S_d is a subset of the L target blocks; the
  dense verifier is S_d = empty.
* Sec. "Domain-to-Configuration Mapping": Phi maps a domain to its skip set; each record carries
  the sparsity ratio R_d = |S_d| / L.
* Sec. "Domain-Aware Skip Controller", first equation: S(x) = Phi(d(x)) for a supported domain,
  the empty set otherwise; fixed for the whole request.
* Same section, second equation: h_{l+1} = f_l(h_l) for l not in S(x), h_{l+1} = h_l for l in
  S(x); a skipped block does neither attention nor feed-forward work (and so writes no KV).
* App. "Models": f_l is a LLaMA block (RMSNorm, rotary multi-head attention, SwiGLU MLP).
* Sec. "Models and speculative decoding methods": the accept/reject rule is the base method's,
  unchanged; the evaluation uses temperature 0 (greedy).  The stochastic rule is the speculative
  sampling of the works the paper cites for speculative decoding (Leviathan et al. 2023,
  Chen et al. 2023).

Readings of points the paper leaves open:
* layer indices are 0-based; RoPE uses the "rotate-half" pairing (i, i + D/2) with
  inv_freq_i = theta^(-2i/D), angles in float64;
* new K and V rows are rounded to bf16 before they are stored or attended (storage precision);
* a draft block is [root = last committed token, draft nodes...]; row i attends to every context
  key and to block rows that are its ancestors or itself;
* argmax ties go to the lowest token id; tree acceptance takes the lowest-index matching child.

Arithmetic runs in the dtype passed as ``dt`` (float32 by default, float64 for the pins).
Weights may be given as float arrays or as uint16 arrays holding bf16 bit patterns.

Parity status: every function is pinned by tests/test_oracle_*.py (closed forms, brute force,
invariants and the published Philox vectors); none is "parity unpinned".
"""
from __future__ import annotations

from typing import Dict, List, Optional, Sequence, Tuple

import numpy as np

from .philox import verify_uniforms

GREEDY_MARGIN = 0.05  # top-2 logit margin below which a greedy decision is flagged
SAMPLE_LOG_BAND = 0.05  # |ln(r q(x)) - ln p(x)| below which an accept test is flagged
SAMPLE_CDF_BAND = 2e-4  # slack (normalised mass) allowed when a drawn token is checked for validity


# ----------------------------------------------------------------------------------------------
# Number formats
# ----------------------------------------------------------------------------------------------
def bf16_bits_to_f32(u16) -> np.ndarray:
    """Exact float32 values of bf16 bit patterns."""
    return (np.asarray(u16, dtype=np.uint16).astype(np.uint32) << np.uint32(16)).view(np.float32)


def round_to_bf16(x) -> np.ndarray:
    """Round to the nearest bf16 value (ties to even) via float32; returned as float32."""
    x = np.ascontiguousarray(x, dtype=np.float32)
    u = x.view(np.uint32).astype(np.uint64)
    r = (u + np.uint64(0x7FFF) + ((u >> np.uint64(16)) & np.uint64(1))) & np.uint64(0xFFFF0000)
    return r.astype(np.uint32).view(np.float32)


def as_float(w, dt=np.float32) -> np.ndarray:
    w = np.asarray(w)
    if w.dtype == np.uint16:
        return bf16_bits_to_f32(w).astype(dt, copy=False)
    return w.astype(dt, copy=False)


# ----------------------------------------------------------------------------------------------
# Skip controller (Sec. "Domain-Aware Skip Controller"; Sec. "Domain-to-Configuration Mapping")
# ----------------------------------------------------------------------------------------------
def skip_set(phi: Dict[int, Sequence[int]], domain: int) -> frozenset:
    """S(x) = Phi(d(x)) if the domain is supported, else the empty set (dense fallback)."""
    if domain in phi:
        return frozenset(int(l) for l in phi[domain])
    return frozenset()


def mask_to_set(mask: int) -> frozenset:
    return frozenset(l for l in range(64) if (int(mask) >> l) & 1)


def set_to_mask(layers) -> int:
    m = 0
    for l in layers:
        m |= 1 << int(l)
    return m


def sparsity_ratio(skip: Sequence[int], n_layers: int) -> float:
    """R_d = |S_d| / L (Sec. "Domain-to-Configuration Mapping")."""
    return len(set(skip)) / float(n_layers)


def active_layers(skip, n_layers: int) -> List[int]:
    """Layers a request runs, in order: {l : l not in S(x)}."""
    return [l for l in range(n_layers) if l not in skip]


def union_active_layers(skips: Sequence[frozenset], n_layers: int) -> List[int]:
    """Layers that at least one request of a batch runs (their weights are read once)."""
    return [l for l in range(n_layers) if any(l not in s for s in skips)]


def layer_row_lists(skips: Sequence[frozenset], n_nodes: Sequence[int], n_layers: int) -> Dict[int, List[int]]:
    """For every layer of the union, the batch rows (requests' rows in batch order) that run it."""
    offs = np.concatenate([[0], np.cumsum(n_nodes)]).astype(int)
    out = {}
    for l in union_active_layers(skips, n_layers):
        rows = []
        for b, s in enumerate(skips):
            if l not in s:
                rows.extend(range(offs[b], offs[b + 1]))
        out[l] = rows
    return out


# ----------------------------------------------------------------------------------------------
# Draft-block structure
# ----------------------------------------------------------------------------------------------
def check_parents(parents: Sequence[int]) -> None:
    if len(parents) == 0 or parents[0] != -1:
        raise ValueError("row 0 must be the root (parent -1)")
    for i, p in enumerate(parents[1:], start=1):
        if not (0 <= p < i):
            raise ValueError(f"parent of row {i} must be in [0, {i})")


def depths(parents: Sequence[int]) -> np.ndarray:
    d = np.zeros(len(parents), dtype=np.int64)
    for i in range(1, len(parents)):
        d[i] = d[parents[i]] + 1
    return d


def ancestor_or_self(parents: Sequence[int]) -> np.ndarray:
    """allowed[i, j] = True iff block row j is row i or one of its ancestors."""
    n = len(parents)
    allowed = np.zeros((n, n), dtype=bool)
    for i in range(n):
        j = i
        while j != -1:
            allowed[i, j] = True
            j = parents[j]
    return allowed


# ----------------------------------------------------------------------------------------------
# LLaMA block pieces (App. "Models")
# ----------------------------------------------------------------------------------------------
def rms_norm(h: np.ndarray, g: np.ndarray, eps: float) -> np.ndarray:
    """h / sqrt(mean(h^2) + eps) * g over the last axis."""
    ms = np.mean(h * h, axis=-1, keepdims=True)
    return h / np.sqrt(ms + eps) * g


def rope_cos_sin(positions, head_dim: int, theta: float, dt=np.float32):
    """cos/sin tables [n, D/2] for angles pos * theta^(-2i/D), computed in float64."""
    half = head_dim // 2
    inv_freq = float(theta) ** (-(2.0 * np.arange(half, dtype=np.float64)) / head_dim)
    ang = np.asarray(positions, dtype=np.float64)[:, None] * inv_freq[None, :]
    return np.cos(ang).astype(dt), np.sin(ang).astype(dt)


def apply_rope(x: np.ndarray, cos: np.ndarray, sin: np.ndarray) -> np.ndarray:
    """Rotate each pair (x_i, x_{i+D/2}) of x [n, H, D] by the angle of its row and index i."""
    half = x.shape[-1] // 2
    x1, x2 = x[..., :half], x[..., half:]
    c, s = cos[:, None, :], sin[:, None, :]
    return np.concatenate([x1 * c - x2 * s, x2 * c + x1 * s], axis=-1)


def silu(x: np.ndarray) -> np.ndarray:
    return x / (1.0 + np.exp(-x))


def block_attention(q, k_ctx, v_ctx, k_blk, v_blk, allowed) -> np.ndarray:
    """Multi-head attention of draft-block queries over context plus allowed block keys.

    q, k_blk, v_blk: [N, H, D]; k_ctx, v_ctx: [H, C, D]; allowed: [N, N] bool.
    Row i attends to all C context keys and to block key j iff allowed[i, j]; scores
    q.k / sqrt(D), softmax with the row maximum subtracted, weights times V.
    """
    N, H, D = q.shape
    C = k_ctx.shape[1]
    out = np.empty_like(q)
    keep = np.concatenate([np.ones((N, C), dtype=bool), allowed], axis=1)
    for h in range(H):
        K = np.concatenate([k_ctx[h], k_blk[:, h, :]], axis=0)
        V = np.concatenate([v_ctx[h], v_blk[:, h, :]], axis=0)
        s = (q[:, h, :] @ K.T) / np.sqrt(q.dtype.type(D))
        s = np.where(keep, s, -np.inf)
        s = s - s.max(axis=1, keepdims=True)
        p = np.exp(s)
        p = p / p.sum(axis=1, keepdims=True)
        out[:, h, :] = p @ V
    return out


def llama_block(h, lw, arch, positions, allowed, k_ctx, v_ctx, dt=np.float32):
    """f_l: one LLaMA block on the draft-block rows h [N, d].

    Returns (h_out, k_new, v_new) with k_new, v_new [N, H, D] rounded to bf16 (the values the
    block stores in its KV cache and attends to).
    """
    N, d = h.shape
    H, D = arch.n_heads, arch.head_dim
    xn = rms_norm(h, as_float(lw["attn_norm"], dt), arch.rms_eps)
    q = (xn @ as_float(lw["wq"], dt).T).reshape(N, H, D)
    k = (xn @ as_float(lw["wk"], dt).T).reshape(N, H, D)
    v = (xn @ as_float(lw["wv"], dt).T).reshape(N, H, D)
    cos, sin = rope_cos_sin(positions, D, arch.rope_theta, dt)
    q = apply_rope(q, cos, sin)
    k = apply_rope(k, cos, sin)
    k = round_to_bf16(k).astype(dt)
    v = round_to_bf16(v).astype(dt)
    o = block_attention(q, k_ctx, v_ctx, k, v, allowed).reshape(N, d)
    h = h + o @ as_float(lw["wo"], dt).T
    xn2 = rms_norm(h, as_float(lw["mlp_norm"], dt), arch.rms_eps)
    g = xn2 @ as_float(lw["w_gate"], dt).T
    u = xn2 @ as_float(lw["w_up"], dt).T
    h = h + (silu(g) * u) @ as_float(lw["w_down"], dt).T
    return h, k, v


def empty_kv(arch, dt=np.float32):
    H, D = arch.n_heads, arch.head_dim
    return np.zeros((H, 0, D), dt), np.zeros((H, 0, D), dt)


def verify_request(weights, arch, skip, tokens, parents, ctx_len: int, kv, dt=np.float32,
                   positions=None, return_hidden=False):
    """Target verification of one request's draft block under skip set ``skip``.

    weights: dict(embed, lm_head, final_norm, layers=[dict per layer]).
    kv: kv[l] = (K [H, >=ctx_len, D], V) holding the request's context for every layer it runs
        (entries of skipped layers are never touched and may be None).
    Returns (logits [N, V], new_kv {l: (k [N,H,D], v [N,H,D])}) and, with return_hidden, the final
    residual [N, d].  Positions default to ctx_len + depth.
    """
    check_parents(parents)
    tokens = np.asarray(tokens, dtype=np.int64)
    if positions is None:
        positions = ctx_len + depths(parents)
    allowed = ancestor_or_self(parents)
    h = as_float(weights["embed"], dt)[tokens]
    new_kv = {}
    for l in range(arch.n_layers):
        if l in skip:
            continue  # h_{l+1} = h_l: no attention, no feed-forward, no KV
        k_ctx = as_float(kv[l][0], dt)[:, :ctx_len, :]
        v_ctx = as_float(kv[l][1], dt)[:, :ctx_len, :]
        h, k, v = llama_block(h, weights["layers"][l], arch, positions, allowed, k_ctx, v_ctx, dt)
        new_kv[l] = (k, v)
    hf = rms_norm(h, as_float(weights["final_norm"], dt), arch.rms_eps)
    logits = hf @ as_float(weights["lm_head"], dt).T
    if return_hidden:
        return logits, new_kv, h
    return logits, new_kv


def verify_requests(weights, arch, skips, blocks, kv, dt=np.float32):
    """verify_request for several requests at once, layer by layer: block b = (tokens, parents,
    ctx_len) runs under skip set skips[b], with context kv(b, l) = (K [H, >=ctx_len, D], V).

    The arithmetic of each request is verify_request's, in the same order, so the results are the
    same; only the loop order differs (layer-major: weights["layers"][l] is read once per batch).
    Returns a list of (logits [N_b, V], new_kv_b).
    """
    h, pos, allowed = [], [], []
    for tokens, parents, ctx_len in blocks:
        check_parents(parents)
        h.append(as_float(weights["embed"], dt)[np.asarray(tokens, dtype=np.int64)])
        pos.append(ctx_len + depths(parents))
        allowed.append(ancestor_or_self(parents))
    new_kv = [{} for _ in blocks]
    for l in range(arch.n_layers):
        runs = [b for b in range(len(blocks)) if l not in skips[b]]
        if not runs:
            continue  # no request runs layer l
        lw = weights["layers"][l]
        for b in runs:
            ctx_len = blocks[b][2]
            k_ctx, v_ctx = kv(b, l)
            k_ctx = as_float(k_ctx, dt)[:, :ctx_len, :]
            v_ctx = as_float(v_ctx, dt)[:, :ctx_len, :]
            h[b], k, v = llama_block(h[b], lw, arch, pos[b], allowed[b], k_ctx, v_ctx, dt)
            new_kv[b][l] = (k, v)
    out = []
    for b in range(len(blocks)):
        hf = rms_norm(h[b], as_float(weights["final_norm"], dt), arch.rms_eps)
        out.append((hf @ as_float(weights["lm_head"], dt).T, new_kv[b]))
    return out


def prefill(weights, arch, skip, ctx_tokens, dt=np.float32):
    """KV of a context under the request's skip set: the causal (chain) forward of the context
    with an empty cache.  Returns kv[l] = (K [H, C, D], V) for active layers, None for skipped."""
    C = len(ctx_tokens)
    parents = [-1] + list(range(C - 1))
    empty = [empty_kv(arch, dt) if l not in skip else None for l in range(arch.n_layers)]
    _, new_kv = verify_request(weights, arch, skip, ctx_tokens, parents, 0, empty, dt)
    kv = [None] * arch.n_layers
    for l, (k, v) in new_kv.items():
        kv[l] = (np.transpose(k, (1, 0, 2)).copy(), np.transpose(v, (1, 0, 2)).copy())
    return kv


def append_kv(kv, new_kv, rows: Sequence[int]):
    """Context KV extended by the block rows ``rows`` (in that order) of every layer in new_kv."""
    out = list(kv)
    rows = list(rows)
    for l, (k, v) in new_kv.items():
        kc, vc = kv[l]
        out[l] = (np.concatenate([kc, np.transpose(k[rows], (1, 0, 2))], axis=1),
                  np.concatenate([vc, np.transpose(v[rows], (1, 0, 2))], axis=1))
    return out


# ----------------------------------------------------------------------------------------------
# Acceptance (temperature 0: greedy; temperature > 0: speculative sampling)
# ----------------------------------------------------------------------------------------------
def argmax_lowest(row) -> int:
    """Index of the largest value; the lowest index among equal maxima."""
    return int(np.argmax(np.asarray(row)))


def top2_margin(row) -> float:
    r = np.asarray(row, dtype=np.float64)
    if r.size < 2:
        return np.inf
    top = np.partition(r, -2)[-2:]
    return float(top[1] - top[0])


def children_of(parents: Sequence[int]) -> List[List[int]]:
    ch = [[] for _ in parents]
    for i, p in enumerate(parents):
        if p >= 0:
            ch[p].append(i)
    return ch


def greedy_accept(logits, tokens, parents) -> Tuple[int, int, List[int]]:
    """Greedy verification of a chain or tree draft.

    Starting at the root, step to the (lowest-index) child whose token equals the argmax of the
    current row, while one exists.  Returns (accept_len a, bonus = argmax of the last row reached,
    path = [0, n_1, ..., n_a]).  For a chain this is the longest prefix with
    draft_i == argmax(row i-1).
    """
    ch = children_of(parents)
    cur = 0
    path = [0]
    while True:
        want = argmax_lowest(logits[cur])
        nxt = next((c for c in ch[cur] if int(tokens[c]) == want), None)
        if nxt is None:
            return len(path) - 1, want, path
        cur = nxt
        path.append(cur)


def greedy_flagged(logits, path, margin: float = GREEDY_MARGIN) -> bool:
    """True if any row the greedy walk read has a top-2 margin below ``margin``."""
    return any(top2_margin(logits[i]) < margin for i in path)


def softmax_t(row, temperature: float, dt=np.float64) -> np.ndarray:
    z = np.asarray(row, dtype=dt) / dt(temperature)
    z = z - z.max()
    e = np.exp(z)
    return e / e.sum()


def inverse_cdf(weights, u: float) -> Tuple[int, float, float, float]:
    """Smallest v with cumsum(weights)[v] > u * sum(weights), by ascending token id.

    Returns (v, target, lower boundary, upper boundary) of v's CDF interval."""
    c = np.cumsum(np.asarray(weights, dtype=np.float64))
    total = c[-1]
    t = u * total
    v = int(np.searchsorted(c, t, side="right"))
    v = min(v, len(c) - 1)
    lo = c[v - 1] if v > 0 else 0.0
    return v, t / total, lo / total, c[v] / total


def uniform_slots(k: int):
    """Slot layout of the uniforms one chain verify uses: r_i (accept test of draft i, i=1..k)
    at slot i-1; u_i (residual draw at draft i, or the bonus draw at i = k+1) at slot k+i-1."""
    return (lambda i: i - 1), (lambda i: k + i - 1), 2 * k + 1


def spec_sample_accept(logits, tokens, q, uniforms, temperature: float = 1.0, return_draw: bool = False):
    """Speculative sampling on a chain draft (rule of the cited speculative-decoding works).

    logits: [k+1, V] target logits of rows 0..k; tokens: [k+1] (row 0 the root);
    q: [k+1, V] draft distributions (row i is the distribution draft token i was sampled from);
    uniforms: [2k+1] laid out as in uniform_slots.
    p_i = softmax(logits_i / T).  For i = 1..k: accept x_i iff r_i * q_i(x_i) < p_{i-1}(x_i)
    (r_i < min(1, p/q) without a division); at the first rejection sample the bonus from
    normalise(max(0, p_{i-1} - q_i)) by inverse CDF with u_i and stop; if all k are accepted
    sample the bonus from p_k with u_{k+1}.
    Returns (a, bonus, path, flagged): flagged marks an accept/reject decision within
    SAMPLE_LOG_BAND of its boundary.  With return_draw, also (weights, u) of the bonus draw.
    """
    k = len(tokens) - 1
    r_slot, u_slot, _ = uniform_slots(k)
    flagged = False
    for i in range(1, k + 1):
        p = softmax_t(logits[i - 1], temperature)
        x = int(tokens[i])
        qx = float(q[i][x])
        if qx <= 0.0:
            raise ValueError("draft token has zero draft probability")
        r = float(uniforms[r_slot(i)])
        lhs, rhs = r * qx, float(p[x])
        if lhs > 0 and rhs > 0 and abs(np.log(lhs) - np.log(rhs)) < SAMPLE_LOG_BAND:
            flagged = True
        if lhs < rhs:
            continue
        res = np.maximum(p - np.asarray(q[i], dtype=np.float64), 0.0)
        u = float(uniforms[u_slot(i)])
        v = inverse_cdf(res, u)[0]
        out = (i - 1, v, list(range(i)), flagged)
        return out + ((res, u),) if return_draw else out
    p = softmax_t(logits[k], temperature)
    u = float(uniforms[u_slot(k + 1)])
    v = inverse_cdf(p, u)[0]
    out = (k, v, list(range(k + 1)), flagged)
    return out + ((p, u),) if return_draw else out


def draw_consistent(weights, u: float, v: int, band: float = SAMPLE_CDF_BAND) -> bool:
    """True if token v is the inverse-CDF draw of u from ``weights`` up to ``band`` of normalised
    mass at its interval edges (a drawn token whose boundary moved by rounding is still valid),
    and v carries positive mass."""
    w = np.asarray(weights, dtype=np.float64)
    if not (0 <= v < len(w)) or w[v] <= 0.0:
        return False
    c = np.cumsum(w) / w.sum()
    lo = c[v - 1] if v > 0 else 0.0
    return lo - band <= u <= c[v] + band


def philox_uniforms(seed: int, offset: int, req: int, k: int):
    """The uniforms of request ``req`` for one chain verify with k drafts (Philox4x32-10)."""
    _, _, n = uniform_slots(k)
    return verify_uniforms(seed, offset, req, n)


# ----------------------------------------------------------------------------------------------
# KV compaction to the accepted path
# ----------------------------------------------------------------------------------------------
def compact_block_rows(rows: np.ndarray, path: Sequence[int]) -> np.ndarray:
    """Block-local KV rows after compaction: row j <- row path[j] for j = 0..a (root stays)."""
    return np.asarray(rows)[list(path)]


def new_ctx_len(ctx_len: int, accept_len: int) -> int:
    """Committed length after a verify: context + root + accepted drafts (the bonus token's KV is
    written when it is the root of the next step)."""
    return ctx_len + 1 + accept_len
