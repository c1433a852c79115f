"""Convenience layer over the C ABI for PyTorch users: owns the KV-cache tensors, builds the batch
and result structures from Python lists, and calls tss_verify.

PyTorch only provides device memory and streams here; all verification work runs in libtss.so.
"""
from __future__ import annotations

from typing import Dict, List, Optional, Sequence

import torch

from . import native, synth


class TssRunner:
    def __init__(self, arch: synth.Arch, weights: Dict, *, n_slots: int, kv_cap: int, max_batch: int = 16,
                 max_rows: int = 256, max_nodes: int = 64, max_domains: int = 64, kv_layers: Optional[Sequence[int]] = None,
                 device: str = "cuda"):
        self.arch = arch
        self.device = device
        self.v = native.Verifier(weights, arch, max_batch=max_batch, max_rows=max_rows, max_nodes=max_nodes,
                                 max_domains=max_domains, max_positions=kv_cap + max_nodes + 1)
        self.n_slots, self.cap = n_slots, kv_cap
        want = range(arch.n_layers) if kv_layers is None else kv_layers
        H, D = arch.n_heads, arch.head_dim
        self.kv: List[Optional[torch.Tensor]] = [None] * arch.n_layers
        for l in want:
            self.kv[l] = torch.zeros((n_slots, 2, H, kv_cap, D), dtype=torch.bfloat16, device=device)
        self.kv_struct = self.v.make_kv([t.data_ptr() if t is not None else None for t in self.kv], n_slots, kv_cap)

    @classmethod
    def for_workload(cls, w: synth.Workload, device: str = "cuda", extra_cap: int = 0) -> "TssRunner":
        """The configuration bench.py times for workload w: seeded weights of the layers some
        request runs (generated on the device), one KV slot per request sized to its context plus
        the draft block (plus extra_cap positions for runs of several steps), synthetic context
        KV, and the workload's skip configurations."""
        a = w.arch
        union = w.active_union()
        max_ctx = max(r.ctx_len for r in w.requests)
        max_n = max(len(r.parents) for r in w.requests)
        weights = synth.make_weights(a, w.seed, device=device, layers=union)
        for l in range(a.n_layers):  # layers no request runs still need (unused) tensors for the ABI
            if weights["layers"][l] is None:
                weights["layers"][l] = {k: torch.zeros(s, dtype=torch.bfloat16, device=device)
                                        for k, s in synth.layer_shapes(a).items()}
        run = cls(a, weights, n_slots=len(w.requests), kv_cap=max_ctx + max_n + 8 + extra_cap, max_batch=len(w.requests),
                  max_rows=max(16, w.n_rows), max_nodes=max_n, kv_layers=union, device=device)
        del weights
        if device != "cpu":
            torch.cuda.empty_cache()
        run.set_phi(w.phi)
        run.fill_synthetic(w)
        return run

    def close(self):
        self.v.close()

    def set_phi(self, phi: Dict[int, int]) -> None:
        for dom, mask in phi.items():
            self.v.set_skip_config(int(dom), int(mask))

    def load_phi(self, path: str) -> Dict[int, int]:
        """Apply the skip configurations of a configuration file (phi_config format) for this
        model's layer count; returns the domain -> bitmask map that was set."""
        from . import phi_config
        phi = phi_config.masks(phi_config.load(path, self.arch.n_layers))
        self.set_phi(phi)
        return phi

    def write_kv(self, layer: int, slot: int, k: torch.Tensor, v: torch.Tensor, pos0: int = 0) -> None:
        """k, v: [H, n, D] values for positions [pos0, pos0 + n)."""
        n = k.shape[1]
        self.kv[layer][slot, 0, :, pos0:pos0 + n] = k.to(self.device, torch.bfloat16)
        self.kv[layer][slot, 1, :, pos0:pos0 + n] = v.to(self.device, torch.bfloat16)

    def fill_synthetic(self, w: synth.Workload, slots: Optional[Sequence[int]] = None) -> None:
        """Synthetic context KV of every request (layers it runs), generated on the device."""
        for b, r in enumerate(w.requests):
            slot = b if slots is None else slots[b]
            mask = w.skip_mask(b)
            for l in range(self.arch.n_layers):
                if (mask >> l) & 1 or self.kv[l] is None:
                    continue
                blk = synth.kv_block(self.arch, l, b, r.ctx_len, w.seed, device=self.device)
                self.kv[l][slot, :, :, :r.ctx_len] = blk

    def alloc_results(self, n_req: int, n_rows: int, path_stride: int = 64, logits: bool = True, host: bool = False):
        dev = "cpu" if host else self.device
        pin = host and torch.cuda.is_available()

        def z(*shape, dtype=torch.int32):
            t = torch.zeros(shape, dtype=dtype, device=dev)
            return t.pin_memory() if pin else t

        out = {"accept_len": z(n_req), "bonus": z(n_req), "path": z(n_req, path_stride), "new_ctx_len": z(n_req),
               "logits": z(n_rows, self.arch.vocab, dtype=torch.float32) if logits else None}
        out["_struct"] = self.v.make_result(out["accept_len"], out["bonus"], out["path"], path_stride,
                                            out["new_ctx_len"], out["logits"])
        return out

    def batch(self, requests: Sequence[synth.Request], *, tokens: Optional[torch.Tensor] = None, slots=None,
              mode: int = native.TSS_MODE_GREEDY, temperature: float = 1.0, draft_probs: Optional[torch.Tensor] = None,
              uniforms: Optional[torch.Tensor] = None, philox_seed: int = 0, philox_offset: int = 0,
              io_host: bool = False):
        toks = [t for r in requests for t in r.tokens]
        if tokens is None:
            tokens = torch.tensor(toks, dtype=torch.int32, device="cpu" if io_host else self.device)
        parents = [p for r in requests for p in r.parents]
        b = self.v.make_batch([len(r.parents) for r in requests], [r.ctx_len for r in requests],
                              [r.domain for r in requests], parents, tokens, kv_slot=slots, mode=mode,
                              temperature=temperature, draft_probs=draft_probs, uniforms=uniforms,
                              uniform_stride=0 if uniforms is None else uniforms.shape[1], philox_seed=philox_seed,
                              philox_offset=philox_offset, io_host=io_host)
        b._tokens = tokens
        return b

    def verify(self, batch, results, stream=None) -> None:
        s = stream if stream is not None else torch.cuda.current_stream().cuda_stream
        self.v.verify(batch, self.kv_struct, results["_struct"], s)

    def prefill(self, prompts: Sequence[Sequence[int]], ctx_lens: Sequence[int], domains: Sequence[int], slots=None,
                stream=None) -> None:
        """Append each request's prompt tokens to its KV cache (tss_prefill) under its domain's
        skip configuration; request b's cache then holds ctx_lens[b] + len(prompts[b]) tokens."""
        toks = torch.tensor([t for pr in prompts for t in pr] or [0], dtype=torch.int32, device=self.device)
        s = stream if stream is not None else torch.cuda.current_stream().cuda_stream
        self.v.prefill([len(pr) for pr in prompts], list(ctx_lens), list(domains), toks, self.kv_struct, kv_slot=slots,
                       stream=s)
        self._prefill_tokens = toks  # alive until the stream has used it

    def verify_grouped(self, batch, results, stream=None, events=None) -> int:
        """tss_verify_grouped: one step per group of requests sharing a skip set; returns the groups."""
        s = stream if stream is not None else torch.cuda.current_stream().cuda_stream
        return self.v.verify_grouped(batch, self.kv_struct, results["_struct"], s, events)

    def sync_status(self, stream=None) -> int:
        s = stream if stream is not None else torch.cuda.current_stream().cuda_stream
        return self.v.sync_status(s)
