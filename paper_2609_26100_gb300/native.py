"""ctypes binding of libtss.so: the C ABI declared in include/tss.h, with the same names.

Argument marshalling only: every step of verification runs in the library's CUDA kernels.  The
binding never falls back to another implementation; if the library is missing it raises.
"""
from __future__ import annotations

import ctypes
import os
from typing import Dict, Optional, Sequence

HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(HERE, "libtss.so")

TSS_OK = 0
TSS_ERR_INVALID_ARG = 1
TSS_ERR_OUT_OF_MEMORY = 2
TSS_ERR_KV_CAPACITY = 3
TSS_ERR_CUDA = 4
TSS_ERR_UNSUPPORTED_ARCH = 5
TSS_ERR_TIMEOUT = 6
TSS_ERR_DEVICE_CHECK = 7
TSS_MODE_GREEDY = 0
TSS_MODE_SAMPLE = 1

EXPORTS = (
    "tss_create", "tss_set_skip_config", "tss_clear_skip_config", "tss_sparsity_ratio",
    "tss_active_layer_count", "tss_verify", "tss_verify_profiled", "tss_prefill", "tss_sync_status", "tss_destroy",
    "tss_linear", "tss_linear_static", "tss_read_trace", "tss_status_string", "tss_last_error",
    "tss_estimate_step_bytes", "tss_persistent_plan", "tss_inject_timeout", "tss_philox_uniforms",
    "tss_linear_static_status", "tss_verify_grouped", "tss_attention_kernel",
)

_P = ctypes.c_void_p
_I32P = ctypes.POINTER(ctypes.c_int32)


class TssArch(ctypes.Structure):
    _fields_ = [(n, ctypes.c_int) for n in ("n_layers", "d_model", "n_heads", "head_dim", "d_mlp", "vocab")] + [
        ("rms_eps", ctypes.c_float), ("rope_theta", ctypes.c_float)] + [
        (n, ctypes.c_int) for n in ("max_batch", "max_rows", "max_nodes", "max_domains", "max_positions")]


class TssWeights(ctypes.Structure):
    _fields_ = [("embed", _P), ("lm_head", _P), ("final_norm", _P)] + [
        (n, ctypes.POINTER(_P)) for n in ("attn_norm", "wq", "wk", "wv", "wo", "mlp_norm", "w_gate", "w_up", "w_down")]


class TssVerifyBatch(ctypes.Structure):
    _fields_ = [
        ("n_req", ctypes.c_int), ("n_nodes", _P), ("ctx_len", _P), ("domain_id", _P), ("kv_slot", _P),
        ("parent_idx", _P), ("positions", _P), ("tokens", _P), ("mode", ctypes.c_int),
        ("temperature", ctypes.c_float), ("draft_probs", _P), ("uniforms", _P), ("uniform_stride", ctypes.c_int),
        ("philox_seed", ctypes.c_uint64), ("philox_offset", ctypes.c_uint64), ("io_host", ctypes.c_int)]


class TssKvCache(ctypes.Structure):
    _fields_ = [("layer", ctypes.POINTER(_P)), ("n_slots", ctypes.c_int), ("cap", ctypes.c_int)]


KERNEL_KINDS = ("controller+embed+norms", "qkv_gemm", "attention", "o_gemm", "gate_up_gemm", "down_gemm",
                "lm_head_gemm", "accept+compact", "verify_persistent")


class TssKernelTimes(ctypes.Structure):
    _fields_ = [("ms", ctypes.c_float * 9), ("launches", ctypes.c_int * 9)]


class TssStepBytes(ctypes.Structure):
    _fields_ = [("weights", ctypes.c_uint64), ("kv_read", ctypes.c_uint64), ("kv_write", ctypes.c_uint64),
                ("total", ctypes.c_uint64), ("active_union", ctypes.c_int)]


class TssPersistentPlanInfo(ctypes.Structure):
    _fields_ = [("fits", ctypes.c_int), ("kps", ctypes.c_int), ("stages", ctypes.c_int), ("attn_splits", ctypes.c_int),
                ("smem_bytes", ctypes.c_uint64)]


class TssVerifyResult(ctypes.Structure):
    _fields_ = [("accept_len", _P), ("bonus", _P), ("path", _P), ("path_stride", ctypes.c_int),
                ("new_ctx_len", _P), ("logits", _P)]


_lib = None


def lib() -> ctypes.CDLL:
    """Load libtss.so (built by __graft_entry__.build() or paper_2609_26100_gb300/build.py)."""
    global _lib
    if _lib is None:
        if not os.path.exists(LIB_PATH):
            raise RuntimeError(f"{LIB_PATH} is missing: build it first (python -c 'import __graft_entry__ as g; g.build()')")
        L = ctypes.CDLL(LIB_PATH)
        L.tss_create.argtypes = [ctypes.POINTER(TssWeights), ctypes.POINTER(TssArch), ctypes.POINTER(_P)]
        L.tss_set_skip_config.argtypes = [_P, ctypes.c_int, ctypes.c_uint64]
        L.tss_clear_skip_config.argtypes = [_P, ctypes.c_int]
        L.tss_sparsity_ratio.argtypes = [_P, ctypes.c_int, ctypes.POINTER(ctypes.c_double)]
        L.tss_active_layer_count.argtypes = [_P, ctypes.POINTER(TssVerifyBatch), ctypes.POINTER(ctypes.c_int)]
        L.tss_verify.argtypes = [_P, ctypes.POINTER(TssVerifyBatch), ctypes.POINTER(TssKvCache),
                                 ctypes.POINTER(TssVerifyResult), _P]
        L.tss_verify_profiled.argtypes = [_P, ctypes.POINTER(TssVerifyBatch), ctypes.POINTER(TssKvCache),
                                          ctypes.POINTER(TssVerifyResult), _P, ctypes.POINTER(TssKernelTimes)]
        L.tss_prefill.argtypes = [_P, ctypes.c_int, _I32P, _I32P, _I32P, _I32P, _P, ctypes.c_int,
                                  ctypes.POINTER(TssKvCache), _P]
        L.tss_sync_status.argtypes = [_P, _P]
        L.tss_destroy.argtypes = [_P]
        L.tss_destroy.restype = None
        L.tss_linear.argtypes = [_P, _P, _P, _P, ctypes.c_int, ctypes.c_int, ctypes.c_int, _P]
        L.tss_linear_static.argtypes = [_P, _P, _P, ctypes.c_int, ctypes.c_int, ctypes.c_int, _P]
        L.tss_read_trace.argtypes = [_P, _P, ctypes.c_size_t, ctypes.POINTER(ctypes.c_size_t)]
        L.tss_status_string.argtypes = [ctypes.c_int]
        L.tss_status_string.restype = ctypes.c_char_p
        L.tss_last_error.argtypes = []
        L.tss_last_error.restype = ctypes.c_char_p
        L.tss_estimate_step_bytes.argtypes = [ctypes.POINTER(TssArch), ctypes.c_int, ctypes.POINTER(ctypes.c_uint64),
                                              _I32P, _I32P, ctypes.POINTER(TssStepBytes)]
        L.tss_persistent_plan.argtypes = [ctypes.POINTER(TssArch), ctypes.c_int, ctypes.c_int, ctypes.c_int,
                                          ctypes.c_int, ctypes.POINTER(TssPersistentPlanInfo)]
        L.tss_inject_timeout.argtypes = [_P, ctypes.c_int]
        L.tss_philox_uniforms.argtypes = [ctypes.c_uint64, ctypes.c_uint64, ctypes.c_int, ctypes.c_int, _P, _P, _P]
        L.tss_linear_static_status.argtypes = [_P]
        L.tss_verify_grouped.argtypes = [_P, ctypes.POINTER(TssVerifyBatch), ctypes.POINTER(TssKvCache),
                                         ctypes.POINTER(TssVerifyResult), _P, ctypes.POINTER(ctypes.c_int),
                                         ctypes.POINTER(_P)]
        L.tss_attention_kernel.argtypes = [_P]
        L.tss_attention_kernel.restype = ctypes.c_int
        for name in ("tss_create", "tss_set_skip_config", "tss_clear_skip_config", "tss_sparsity_ratio",
                     "tss_active_layer_count", "tss_verify", "tss_verify_profiled", "tss_prefill", "tss_sync_status",
                     "tss_linear", "tss_linear_static", "tss_read_trace", "tss_estimate_step_bytes",
                     "tss_persistent_plan", "tss_inject_timeout", "tss_philox_uniforms", "tss_linear_static_status",
                     "tss_verify_grouped"):
            getattr(L, name).restype = ctypes.c_int
        _lib = L
    return _lib


def linear_static(x, w, y, stream=None) -> None:
    """y = x @ w^T through tss_linear_static (no context, no device allocation)."""
    m, k = x.shape
    check(lib().tss_linear_static(x.data_ptr(), w.data_ptr(), y.data_ptr(), m, k, w.shape[0], stream),
          "tss_linear_static")


def linear_static_status(stream=None) -> int:
    """tss_linear_static_status: synchronise, return and clear the static linear layer's status."""
    return lib().tss_linear_static_status(stream)


def philox_uniforms(seed: int, offset: int, words=None, uniforms=None, stream=None) -> None:
    """tss_philox_uniforms into device tensors words [n_req][n_slots][4] (int32 or uint32 bits)
    and/or uniforms [n_req][n_slots] (float32)."""
    t = words if words is not None else uniforms
    n_req, n_slots = int(t.shape[0]), int(t.shape[1])
    check(lib().tss_philox_uniforms(int(seed), int(offset), n_req, n_slots, _ptr(words), _ptr(uniforms), stream),
          "tss_philox_uniforms")


def persistent_plan(arch, n_req: int, n_rows: int, max_keys: int, num_sms: int) -> Dict[str, int]:
    """tss_persistent_plan: the persistent kernel's shared-memory plan for a step (host only)."""
    a = TssArch(arch.n_layers, arch.d_model, arch.n_heads, arch.head_dim, arch.d_mlp, arch.vocab,
                arch.rms_eps, arch.rope_theta, 1, 1, 1, 1, 1)
    out = TssPersistentPlanInfo()
    check(lib().tss_persistent_plan(ctypes.byref(a), n_req, n_rows, max_keys, num_sms, ctypes.byref(out)),
          "tss_persistent_plan")
    return {"fits": bool(out.fits), "kps": out.kps, "stages": out.stages, "attn_splits": out.attn_splits,
            "smem_bytes": out.smem_bytes}


def estimate_step_bytes(arch, masks: Sequence[int], ctx_len: Sequence[int], n_nodes: Sequence[int]) -> Dict[str, int]:
    """tss_estimate_step_bytes: HBM bytes of a verification step (host arithmetic, no GPU)."""
    a = TssArch(arch.n_layers, arch.d_model, arch.n_heads, arch.head_dim, arch.d_mlp, arch.vocab,
                arch.rms_eps, arch.rope_theta, 1, 1, 1, 1, 1)
    n = len(masks)
    m = (ctypes.c_uint64 * n)(*[int(x) for x in masks])
    out = TssStepBytes()
    check(lib().tss_estimate_step_bytes(ctypes.byref(a), n, m, ctypes.cast(_i32(ctx_len), _I32P),
                                        ctypes.cast(_i32(n_nodes), _I32P), ctypes.byref(out)), "tss_estimate_step_bytes")
    return {"weights": out.weights, "kv_read": out.kv_read, "kv_write": out.kv_write, "total": out.total,
            "active_union": out.active_union}


class TssError(RuntimeError):
    def __init__(self, status: int, where: str):
        L = lib()
        self.status = status
        msg = L.tss_last_error().decode()
        super().__init__(f"{where}: {L.tss_status_string(status).decode()} ({status}): {msg}")


def check(status: int, where: str) -> None:
    if status != TSS_OK:
        raise TssError(status, where)


def _ptr(t) -> Optional[int]:
    """Address of a tensor / numpy array (None -> NULL)."""
    if t is None:
        return None
    if hasattr(t, "data_ptr"):
        return t.data_ptr()
    return t.ctypes.data


def _i32(values) -> "ctypes.Array":
    arr = (ctypes.c_int32 * len(values))(*[int(v) for v in values])
    return arr


class Verifier:
    """Owns one tss_ctx.  Weights: dict as produced by synth.make_weights (bf16 CUDA tensors)."""

    def __init__(self, weights: Dict, arch, max_batch: int = 16, max_rows: int = 256, max_nodes: int = 64,
                 max_domains: int = 64, max_positions: int = 20480):
        L = lib()
        self.arch = arch
        a = TssArch(arch.n_layers, arch.d_model, arch.n_heads, arch.head_dim, arch.d_mlp, arch.vocab,
                    arch.rms_eps, arch.rope_theta, max_batch, max_rows, max_nodes, max_domains, max_positions)
        self._arch = a
        n = arch.n_layers
        arrs = {}
        for key in ("attn_norm", "wq", "wk", "wv", "wo", "mlp_norm", "w_gate", "w_up", "w_down"):
            arrs[key] = (_P * n)(*[weights["layers"][l][key].data_ptr() for l in range(n)])
        w = TssWeights(weights["embed"].data_ptr(), weights["lm_head"].data_ptr(), weights["final_norm"].data_ptr(),
                       *[ctypes.cast(arrs[k], ctypes.POINTER(_P)) for k in
                         ("attn_norm", "wq", "wk", "wv", "wo", "mlp_norm", "w_gate", "w_up", "w_down")])
        h = _P()
        check(L.tss_create(ctypes.byref(w), ctypes.byref(a), ctypes.byref(h)), "tss_create")
        self.ctx = h

    def close(self):
        if getattr(self, "ctx", None):
            lib().tss_destroy(self.ctx)
            self.ctx = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    def set_skip_config(self, domain: int, mask: int) -> None:
        check(lib().tss_set_skip_config(self.ctx, domain, mask), "tss_set_skip_config")

    def clear_skip_config(self, domain: int) -> None:
        check(lib().tss_clear_skip_config(self.ctx, domain), "tss_clear_skip_config")

    def sparsity_ratio(self, domain: int) -> float:
        out = ctypes.c_double()
        check(lib().tss_sparsity_ratio(self.ctx, domain, ctypes.byref(out)), "tss_sparsity_ratio")
        return out.value

    def sync_status(self, stream=None) -> int:
        return lib().tss_sync_status(self.ctx, stream)

    def attention_kernel(self) -> int:
        """tss_attention_kernel: the attention kernel of the last step (0 split-KV warp-MMA kernel,
        1 tcgen05 kernel, 2 its wide variant, 3 inside the persistent kernel, -1 none yet)."""
        return int(lib().tss_attention_kernel(self.ctx))

    def inject_timeout(self, n_steps: int) -> None:
        check(lib().tss_inject_timeout(self.ctx, n_steps), "tss_inject_timeout")

    def linear(self, x, w, y, stream=None) -> None:
        m, k = x.shape
        n = w.shape[0]
        check(lib().tss_linear(self.ctx, x.data_ptr(), w.data_ptr(), y.data_ptr(), m, k, n, stream), "tss_linear")

    @staticmethod
    def make_batch(n_nodes: Sequence[int], ctx_len: Sequence[int], domain_id: Sequence[int], parent_idx: Sequence[int],
                   tokens, kv_slot=None, positions=None, mode: int = TSS_MODE_GREEDY, temperature: float = 1.0,
                   draft_probs=None, uniforms=None, uniform_stride: int = 0, philox_seed: int = 0,
                   philox_offset: int = 0, io_host: bool = False):
        """Build a TssVerifyBatch; host metadata arrays are kept alive on the returned object."""
        keep = {"n_nodes": _i32(n_nodes), "ctx_len": _i32(ctx_len), "domain_id": _i32(domain_id),
                "parent_idx": _i32(parent_idx)}
        if kv_slot is not None:
            keep["kv_slot"] = _i32(kv_slot)
        if positions is not None:
            keep["positions"] = _i32(positions)
        addr = {k: ctypes.cast(v, _P) for k, v in keep.items()}
        b = TssVerifyBatch(
            len(n_nodes), addr["n_nodes"], addr["ctx_len"], addr["domain_id"], addr.get("kv_slot"),
            addr["parent_idx"], addr.get("positions"), _ptr(tokens), mode, temperature, _ptr(draft_probs),
            _ptr(uniforms), uniform_stride, philox_seed, philox_offset, 1 if io_host else 0)
        b._keep = (keep, tokens, draft_probs, uniforms)
        return b

    def make_kv(self, layer_ptrs: Sequence[Optional[int]], n_slots: int, cap: int):
        arr = (_P * len(layer_ptrs))(*[p if p else None for p in layer_ptrs])
        kv = TssKvCache(ctypes.cast(arr, ctypes.POINTER(_P)), n_slots, cap)
        kv._keep = arr
        return kv

    @staticmethod
    def make_result(accept_len, bonus, path, path_stride: int, new_ctx_len, logits=None):
        r = TssVerifyResult(_ptr(accept_len), _ptr(bonus), _ptr(path), path_stride, _ptr(new_ctx_len), _ptr(logits))
        r._keep = (accept_len, bonus, path, new_ctx_len, logits)
        return r

    def verify(self, batch, kv, result, stream=None) -> None:
        check(lib().tss_verify(self.ctx, ctypes.byref(batch), ctypes.byref(kv), ctypes.byref(result), stream),
              "tss_verify")

    def verify_grouped(self, batch, kv, result, stream=None, events=None) -> int:
        """tss_verify_grouped; events: optional list of torch.cuda.Event (one per request, the first
        n_groups are recorded).  Returns the number of groups."""
        n = ctypes.c_int()
        ev = None
        if events is not None:
            for e in events:  # torch creates an event at its first record
                if e is not None and not e.cuda_event:
                    e.record()
            ev = (_P * len(events))(*[e.cuda_event if e is not None else None for e in events])
        check(lib().tss_verify_grouped(self.ctx, ctypes.byref(batch), ctypes.byref(kv), ctypes.byref(result), stream,
                                       ctypes.byref(n), ev), "tss_verify_grouped")
        return n.value

    def prefill(self, n_tokens: Sequence[int], ctx_len: Sequence[int], domain_id: Sequence[int], tokens, kv,
                kv_slot=None, io_host: bool = False, stream=None) -> None:
        """tss_prefill: tokens (int32, the requests' tokens concatenated) appended to the caches."""
        keep = [_i32(n_tokens), _i32(ctx_len), _i32(domain_id), _i32(kv_slot) if kv_slot is not None else None]
        cast = [ctypes.cast(a, _I32P) if a is not None else None for a in keep]
        check(lib().tss_prefill(self.ctx, len(n_tokens), cast[0], cast[1], cast[2], cast[3], _ptr(tokens),
                                1 if io_host else 0, ctypes.byref(kv), stream), "tss_prefill")

    def verify_profiled(self, batch, kv, result, times: "TssKernelTimes", stream=None) -> None:
        check(lib().tss_verify_profiled(self.ctx, ctypes.byref(batch), ctypes.byref(kv), ctypes.byref(result), stream,
                                        ctypes.byref(times)), "tss_verify_profiled")

    def read_trace(self):
        """Persistent-kernel timeline of the last step (see tss_read_trace), as a numpy array
        [n_sms, slots] of globaltimer ns, or None when tracing is off."""
        import numpy as np
        n = ctypes.c_size_t()
        check(lib().tss_read_trace(self.ctx, None, 0, ctypes.byref(n)), "tss_read_trace")
        if n.value == 0:
            return None
        buf = np.zeros(n.value, dtype=np.uint64)
        check(lib().tss_read_trace(self.ctx, buf.ctypes.data, n.value, ctypes.byref(n)), "tss_read_trace")
        return buf

    def active_layer_count(self, batch) -> int:
        out = ctypes.c_int()
        check(lib().tss_active_layer_count(self.ctx, ctypes.byref(batch), ctypes.byref(out)), "tss_active_layer_count")
        return out.value
