#!/usr/bin/env python
"""Verify-step benchmark of the TSS target-side verification path on GB300.

Default workload: Llama-2-7B-shaped decoder (32 layers, d 4096, 32 x 128 heads, MLP 11008,
vocab 32000), random-init bf16 weights, batch 1, context 1024 (synthetic KV), chain draft k = 5
(uniform random ids; 20% of steps start with a greedy prefix of length 0-5), skip set
{20, 24, 27, 30}, greedy acceptance.  One step = one tss_verify (controller, embedding, every
active layer, LM head + argmax, acceptance, KV compaction).

Prints one JSON line (rank 0).  `value` is verified tokens/s (rows scored per second, B*(k+1)
per step) with inputs resident in HBM; `e2e` is the same metric through the C ABI with host
buffers (token upload and result read-back inside the timed region, one synchronisation per
step).  `--impl reference` times the CPU oracle on a bounded sample of the same workload.
"""
import argparse
import json
import os
import statistics
import subprocess
import sys
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

METRIC = "7B verify-step latency (us) & tokens/s at k=5, 4 skipped layers; % HBM roofline"
# Bytes of the per-step descriptor tss_verify copies to the device (sizeof(tss::StepDesc);
# tests/test_step_bytes.py compiles the struct and checks this number).
STEP_DESC_BYTES = 9840
NOMINAL_HBM_GBS = 8000.0


def parse_args():
    p = argparse.ArgumentParser()
    p.add_argument("--gpus", type=int, default=1)
    p.add_argument("--steps", type=int, default=200)
    p.add_argument("--warmup", type=int, default=10)
    p.add_argument("--impl", default="tss", choices=["tss", "reference"])
    p.add_argument("--workload", default="7b_chain", choices=["7b_chain", "7b_dense", "7b_tree", "13b_mixed", "7b_long", "tiny"])
    p.add_argument("--skip", type=int, default=None, help="7b_long: number of skipped layers (sweep point)")
    p.add_argument("--layers", type=int, default=None,
                   help="truncate the model to its first N layers (small profiling case; not a bench workload)")
    p.add_argument("--no-cpu-baseline", action="store_true")
    p.add_argument("--no-e2e", action="store_true")
    p.add_argument("--no-profile", action="store_true")
    p.add_argument("--sweep", default=None,
                   help="7b_long or 7b_chain: comma-separated skipped-layer counts (e.g. 0,2,4,...,12); one "
                        "process, one weight and KV set, latency vs active layers with a least-squares line")
    p.add_argument("--prefill", type=int, default=None,
                   help="prompt tokens per request: time tss_prefill on the 7B chain's skip set (4 requests) "
                        "instead of the verification step")
    p.add_argument("--grouped", action="store_true",
                   help="time tss_verify_grouped (one step per skip set, fewest active layers first) against the "
                        "mixed step on the workload (13b_mixed by default): per-request completion times")
    p.add_argument("--traffic", default=os.path.join(ROOT, "profiles"),
                   help="JSON summary of an ncu DRAM-traffic capture of the dominant kernel, or a directory "
                        "whose *_traffic.txt files are such summaries")
    return p.parse_args()


def make_workload(name, skip=None):
    from paper_2609_26100_gb300 import synth
    if name == "7b_chain":
        return synth.workload_7b_chain()
    if name == "7b_dense":
        return synth.workload_7b_chain(mask_layers=())
    if name == "7b_tree":
        return synth.workload_7b_tree()
    if name == "13b_mixed":
        return synth.workload_13b_mixed()
    if name == "7b_long":
        return synth.workload_7b_long(n_skip=8 if skip is None else skip)
    if name == "tiny":
        return synth.config_chain(synth.TINY, "tiny_bench", 1, [128], 4, {0: synth.mask_of([2])}, [0])
    raise ValueError(name)


def workload_config(w, args):
    a = w.arch
    ks = sorted({len(r.parents) - 1 for r in w.requests})
    return {
        "workload": f"{w.name}: L{a.n_layers} d{a.d_model} H{a.n_heads}x{a.head_dim} F{a.d_mlp} V{a.vocab}, "
                    f"B={len(w.requests)}, ctx={sorted({r.ctx_len for r in w.requests})[:4]}, "
                    f"rows={w.n_rows}, k={ks}, active_union={len(w.active_union())}/{a.n_layers}, mode={w.mode}",
        "batch": len(w.requests), "rows_per_step": w.n_rows,
        "skip_sets": {str(d): [l for l in range(64) if (m >> l) & 1] for d, m in w.phi.items()},
        "parallelism": f"replicas x{args.gpus}" if args.gpus > 1 else "single GPU",
        "l2": "inputs larger than L2: every step streams the active-layer weights (GBs) from HBM",
    }


def measured_peak():
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            pk = json.load(f)
        return float(pk["hbm_gbs"]), "measured"
    except Exception:
        return 6800.0, "fallback"


class ClockSampler:
    """nvidia-smi samples of this GPU's clocks and throttle reasons during the timed region."""
    FIELDS = ("pci.bus_id,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, bus_id):
        self.bus_id = bus_id.lower()
        self.proc = None

    def __enter__(self):
        try:
            self.proc = subprocess.Popen(["nvidia-smi", f"--query-gpu={self.FIELDS}", "--format=csv,noheader,nounits",
                                          "-lms", "200"], stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except Exception:
            self.proc = None
        time.sleep(0.3)
        return self

    def __exit__(self, *exc):
        self.out = ""
        if self.proc:
            self.proc.terminate()
            try:
                self.out, _ = self.proc.communicate(timeout=5)
            except Exception:
                self.proc.kill()
        return False

    def summary(self):
        rows = []
        for ln in (self.out or "").splitlines():
            f = [x.strip() for x in ln.split(",")]
            if len(f) < 9:
                continue
            if self.bus_id and not f[0].lower().endswith(self.bus_id[-12:]):
                continue
            rows.append(f)
        if not rows:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["no nvidia-smi samples"], "samples": 0}
        sm = [float(r[1]) for r in rows if r[1].replace(".", "").isdigit()]
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({names[i] for r in rows for i in range(4) if r[5 + i].lower() == "active"})
        return {"sm_mhz": statistics.median(sm) if sm else None,
                "sm_max_mhz": float(rows[0][2]) if rows[0][2].replace(".", "").isdigit() else None,
                "reasons": reasons, "samples": len(rows),
                "power_w_max": max(float(r[3]) for r in rows if r[3].replace(".", "").isdigit())}


# Sources of each kernel kind whose ncu traffic figure bench.py may reuse.
KERNEL_SOURCES = {
    "verify_persistent": ("verify_mk.cu", "attn_body.cuh", "common.cuh", "internal.h"),
    "attention": ("attention.cu", "attn_body.cuh", "common.cuh", "internal.h"),
    "attention_tc": ("attn_tc.cu", "common.cuh", "internal.h"),
}

# tss_attention_kernel -> the KERNEL_SOURCES entry of the separate attention kernel that ran
ATTENTION_IMPL = {0: "attention", 1: "attention_tc", 2: "attention"}


def kernel_sources_hash(kernel="verify_persistent"):
    """sha256 over the code of a kernel's sources, comments and blank lines left out (an ncu
    traffic figure is only valid for the kernel it was taken on)."""
    import hashlib
    import re
    h = hashlib.sha256()
    for f in KERNEL_SOURCES[kernel]:
        with open(os.path.join(ROOT, "paper_2609_26100_gb300", "csrc", f), encoding="utf-8") as fh:
            for line in fh:
                code = re.sub(r"(^|\s)//.*$", "", line.rstrip("\n")).rstrip()
                if code:
                    h.update(code.encode() + b"\n")
    return h.hexdigest()


def find_traffic(path, kernel, workload):
    """DRAM bytes per launch of `kernel` on `workload` from an ncu capture summary (JSON with
    "kernel", "workload", "traffic_bytes" and "sources_sha256", the hash of the kernel sources
    it was taken on); None unless one matches the workload and the unchanged sources."""
    import glob
    if not path or not os.path.exists(path) or kernel not in KERNEL_SOURCES:
        return None
    files = sorted(glob.glob(os.path.join(path, "*_traffic.txt"))) if os.path.isdir(path) else [path]
    for fn in files:
        with open(fn) as f:
            tr = json.load(f)
        if (tr.get("kernel") == kernel and tr.get("workload") == workload
                and tr.get("sources_sha256") == kernel_sources_hash(kernel)):
            return tr
    return None


def kernel_bytes(w, kinds):
    """Algorithmic bytes per STEP of each kernel kind present (weights + activations + KV).
    Persistent path: the persistent kernel streams every active layer's weights and the LM head
    (and the KV too when the attention runs inside it); with separate attention launches (long
    contexts) the attention kind carries the KV reads.  Kernel-per-op path: the per-layer
    formulas times the launches."""
    from paper_2609_26100_gb300 import synth
    a = w.arch
    d, f, V, M = a.d_model, a.d_mlp, a.vocab, w.n_rows
    ab = synth.algorithmic_bytes(w)
    kv_read = sum(r.ctx_len for r in w.requests) * a.kv_bytes_per_token  # per layer, all requests
    out = {}
    if "verify_persistent" in kinds:
        if "attention" in kinds:
            out["verify_persistent"] = ab["total"] - ab["kv_read"]
            out["attention"] = ab["kv_read"]
        else:
            out["verify_persistent"] = ab["total"]
        return out
    per_launch = {
        "qkv_gemm": 3 * d * d * 2 + M * d * 2 + M * d * 2 + M * 2 * d * 2,
        "attention": kv_read + M * d * 2 * 2 + M * 2 * d * 2,
        "o_gemm": d * d * 2 + M * d * 2 + M * d * 4 * 2,
        "gate_up_gemm": 2 * f * d * 2 + M * d * 2 + M * f * 2,
        "down_gemm": d * f * 2 + M * f * 2 + M * d * 4 * 2,
        "lm_head_gemm": V * d * 2 + M * d * 2 + M * V * 4,
    }
    for k, v in kinds.items():
        if k in per_launch:
            out[k] = per_launch[k] * v
    return out


# ----------------------------------------------------------------------------------------------
# CPU oracle (cpu_baseline leg and --impl reference)
# ----------------------------------------------------------------------------------------------
def host_mem_available():
    try:
        with open("/proc/meminfo") as f:
            for ln in f:
                if ln.startswith("MemAvailable:"):
                    return int(ln.split()[1]) * 1024
    except OSError:
        pass
    return 0


def cpu_model():
    try:
        out = subprocess.run(["lscpu"], capture_output=True, text=True, timeout=10).stdout
        for ln in out.splitlines():
            if ln.startswith("Model name:"):
                return ln.split(":", 1)[1].strip()
    except Exception:
        pass
    return "unknown"


class OracleStep:
    """The oracle timed on WHOLE verification steps of the workload: every request through
    O.verify_requests (embedding, every layer it runs, final norm, LM head) and the acceptance
    rule, one step per call.  The fp32 weights of the active layers and the requests' context KV
    are generated (seeded, as the GPU run's) before any timing and stay in host memory, so a timed
    step is the oracle's arithmetic only.  Raises MemoryError when they would take more than half
    of the host's available memory."""

    @staticmethod
    def host_bytes(w):
        a = w.arch
        per_layer = 4 * (4 * a.d_model * a.d_model + 3 * a.d_model * a.d_mlp)
        kv = sum(r.ctx_len * len([l for l in range(a.n_layers) if not (w.skip_mask(b) >> l) & 1])
                 for b, r in enumerate(w.requests)) * 2 * a.d_model * 4
        return len(w.active_union()) * per_layer + 2 * a.vocab * a.d_model * 4 + kv

    def __init__(self, w, device):
        from paper_2609_26100_gb300 import synth
        if self.host_bytes(w) > 0.5 * host_mem_available():
            raise MemoryError(f"oracle step needs {self.host_bytes(w) / 1e9:.1f} GB of host memory")
        self.w = w
        a = w.arch
        f32 = lambda t: t.float().cpu().numpy()  # noqa: E731
        g = synth.make_weights(a, w.seed, device=device, layers=[])
        layers = [None] * a.n_layers
        for l in w.active_union():
            layers[l] = {k: f32(v) for k, v in synth.make_layer(a, l, w.seed, device=device).items()}
        self.weights = {"embed": f32(g["embed"]), "lm_head": f32(g["lm_head"]), "final_norm": f32(g["final_norm"]),
                        "layers": layers}
        del g
        self.skips = [frozenset(synth.layers_of(w.skip_mask(b))) for b in range(len(w.requests))]
        self.kv = {}
        for b, r in enumerate(w.requests):
            for l in range(a.n_layers):
                if l not in self.skips[b]:
                    blk = f32(synth.kv_block(a, l, b, r.ctx_len, w.seed, device=device))
                    self.kv[(b, l)] = (blk[0], blk[1])
        if device != "cpu":
            import torch
            torch.cuda.empty_cache()

    def step_seconds(self, i=0):
        from oracle import tss_oracle as O
        w = self.w
        t = time.perf_counter()
        outs = O.verify_requests(self.weights, w.arch, self.skips,
                                 [(r.tokens, r.parents, r.ctx_len) for r in w.requests], lambda b, l: self.kv[(b, l)])
        for b, r in enumerate(w.requests):
            if w.mode == "sample":
                u = O.philox_uniforms(w.seed, i, b, len(r.parents) - 1)
                O.spec_sample_accept(outs[b][0], r.tokens, r.draft_probs.numpy(), u, w.temperature)
            else:
                O.greedy_accept(outs[b][0], r.tokens, r.parents)
        return time.perf_counter() - t

    def describe(self, n):
        w = self.w
        return (f"oracle (NumPy fp32) on whole verification steps of the workload ({len(w.requests)} request(s), "
                f"{len(w.active_union())} active layers, {w.n_rows} rows, acceptance included), weights and context "
                f"KV resident in host memory; median of {n} timed step(s); CPU {cpu_model()}")


def make_oracle(w, device):
    """Whole timed steps when their weights and KV fit in host memory, else the extrapolated sample."""
    try:
        return OracleStep(w, device)
    except MemoryError:
        return OracleSample(w, device)


class OracleSample:
    """The oracle on a bounded sample of the workload: embedding + LM head with every layer
    skipped (t0), and with one sampled active layer (t1); a full step is estimated as
    t0 + n_active * (t1 - t0)."""

    def __init__(self, w, device):
        import numpy as np
        import torch
        from paper_2609_26100_gb300 import synth
        self.w = w
        a = w.arch
        self.union = w.active_union()
        self.sample_layers = self.union[:2]
        gen = synth.make_weights(a, w.seed, device=device, layers=self.sample_layers)
        f32 = lambda t: t.float().cpu().numpy()  # noqa: E731
        self.weights = {"embed": f32(gen["embed"]), "lm_head": f32(gen["lm_head"]), "final_norm": f32(gen["final_norm"]),
                        "layers": [None if lw is None else {k: f32(v) for k, v in lw.items()} for lw in gen["layers"]]}
        del gen
        r = w.requests[0]
        self.kv = [None] * a.n_layers
        for l in self.sample_layers:
            blk = synth.kv_block(a, l, 0, r.ctx_len, w.seed, device=device).float().cpu().numpy()
            self.kv[l] = (blk[0], blk[1])
        if device != "cpu":
            torch.cuda.empty_cache()
        self.np = np

    def _run(self, active):
        from oracle import tss_oracle as O
        a, r = self.w.arch, self.w.requests[0]
        skip = frozenset(l for l in range(a.n_layers) if l not in active)
        t = time.perf_counter()
        O.verify_request(self.weights, a, skip, r.tokens, r.parents, r.ctx_len, self.kv)
        return time.perf_counter() - t

    def step_seconds(self, i=0):
        """Estimated oracle seconds for one full step of request 0 (median-free single sample)."""
        if not hasattr(self, "t0"):
            self.t0 = min(self._run([]) for _ in range(2))
        t1 = self._run([self.sample_layers[i % len(self.sample_layers)]])
        n_act = sum(1 for l in range(self.w.arch.n_layers) if not (self.w.skip_mask(0) >> l) & 1)
        per_req = self.t0 + n_act * max(t1 - self.t0, 0.0)
        return per_req * len(self.w.requests)

    def describe(self, n):
        return (f"EXTRAPOLATED (the workload's weights and KV do not fit in host memory): oracle (NumPy fp32) verify "
                f"of request 0 with all layers skipped and with 1 sampled active layer, extrapolated to its active "
                f"layers and scaled by the batch; {n} sample(s); CPU {cpu_model()}")


def cores():
    try:
        return len(os.sched_getaffinity(0))
    except Exception:
        return os.cpu_count()


# ----------------------------------------------------------------------------------------------
def max_over_ranks(ms, device):
    """The job's time for a timed region: the slowest rank's (every rank gets it).  One process per
    GPU, each timing its own replica; without an initialised process group this is `ms`."""
    import torch
    import torch.distributed as dist
    if not (dist.is_available() and dist.is_initialized()) or dist.get_world_size() == 1:
        return ms
    t = torch.tensor([ms], device=device, dtype=torch.float64)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def job_tokens_per_s(rows_per_step, steps, world, max_ms):
    """Whole-job throughput: every rank verified rows_per_step rows in each of `steps` steps, and
    the job took the slowest rank's time (weak scaling: per-GPU work fixed)."""
    return world * rows_per_step * steps / (max_ms / 1e3)


def run_reference(args):
    rank = int(os.environ.get("RANK", "0"))
    if rank != 0:
        return
    import torch
    w = make_workload(args.workload, args.skip)
    dev = "cuda" if torch.cuda.is_available() else "cpu"
    s = make_oracle(w, dev)
    for i in range(args.warmup):
        s.step_seconds(i)
    times = [s.step_seconds(i) for i in range(args.steps)]
    sec = statistics.median(times)
    value = w.n_rows / sec
    cb = {"value": value, "unit": "tokens/s", "cores": cores(), "kind": "oracle", "sample": s.describe(args.steps),
          "measured": isinstance(s, OracleStep), "timed_s_total": sum(times)}
    print(json.dumps({
        "impl": "reference", "metric": METRIC, "value": value, "unit": "tokens/s", "n_gpus": args.gpus,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": sec * 1e3, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "f32", "data": "synthetic",
        "config": workload_config(w, args), "cpu_baseline": cb,
        "e2e": {"value": value, "unit": "tokens/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}))


def run_tss(args):
    import torch
    import torch.distributed as dist

    from paper_2609_26100_gb300 import build as _build
    from paper_2609_26100_gb300 import native, synth
    from paper_2609_26100_gb300.runner import TssRunner

    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    torch.cuda.set_device(local)
    if world > 1:
        dist.init_process_group("nccl", device_id=torch.device("cuda", local))
    if rank == 0 or world == 1:
        _build.build()
    if world > 1:
        dist.barrier()
    _build.build()  # no-op when up to date
    w = make_workload(args.workload, args.skip)
    if args.layers:
        import dataclasses
        w.arch = dataclasses.replace(w.arch, n_layers=args.layers)
        w.phi = {d: m & ((1 << args.layers) - 1) for d, m in w.phi.items()}
    a = w.arch
    union = w.active_union()

    # cpu baseline sample needs host copies of a few layers; take them before the GPU run
    sample = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        sample = make_oracle(w, "cuda")

    run = TssRunner.for_workload(w)
    stream = torch.cuda.current_stream()

    # Per-step drafts.  7B chain: 20% of steps carry a greedy prefix of length 0-5, built from the
    # model's own greedy continuation (obtained through the library during setup).
    sample_mode = w.mode == "sample"
    probs = None
    if sample_mode:
        probs = torch.cat([r.draft_probs for r in w.requests], 0).cuda()
    n_var = 10
    token_sets = []
    for v in range(n_var):
        toks = []
        for b, r in enumerate(w.requests):
            if sample_mode or v == 0:
                toks.extend(r.tokens)
            else:
                toks.extend(synth.draft_tokens(r.parents, a.vocab, w.seed + v, f"bench.{v}.{b}"))
        token_sets.append(toks)
    if w.name == "7b_chain":
        r = w.requests[0]
        greedy = []
        res = run.alloc_results(1, w.n_rows, logits=False)
        toks = list(token_sets[0])
        for i in range(len(r.parents) - 1):
            b = run.batch([synth.Request(r.ctx_len, r.parents, toks, r.domain)])
            run.verify(b, res)
            torch.cuda.synchronize()
            g = int(res["bonus"][0])
            greedy.append(g)
            toks[i + 1] = g
        sel = synth.uniform_ints(n_var, 5, w.seed, "bench.prefix").tolist()
        for v in range(n_var):
            if v % 5 == 4:  # one step in five: variant 0's root followed by its greedy continuation
                lp = sel[v] + 1
                token_sets[v][0] = token_sets[0][0]
                token_sets[v][1:1 + lp] = greedy[:lp]
    batches = []
    for v in range(n_var):
        tt = torch.tensor(token_sets[v], dtype=torch.int32, device="cuda")
        batches.append(run.batch(w.requests, tokens=tt,
                                 mode=native.TSS_MODE_SAMPLE if sample_mode else native.TSS_MODE_GREEDY,
                                 temperature=w.temperature, draft_probs=probs, philox_seed=w.seed, philox_offset=v))
    res = run.alloc_results(len(w.requests), w.n_rows, logits=False)
    for i in range(args.warmup):
        run.verify(batches[i % n_var], res)
    if run.sync_status() != native.TSS_OK:
        raise RuntimeError("device status error during warm-up")

    # ---------------- timed region (device-resident inputs) ----------------
    ev = [torch.cuda.Event(enable_timing=True) for _ in range(args.steps + 1)]
    bus = torch.cuda.get_device_properties(local).pci_bus_id if hasattr(torch.cuda.get_device_properties(local), "pci_bus_id") else ""
    if world > 1:
        dist.barrier()
    torch.cuda.synchronize()
    with ClockSampler(str(bus)) as clk:
        ev[0].record(stream)
        for i in range(args.steps):
            run.verify(batches[i % n_var], res)
            ev[i + 1].record(stream)
        torch.cuda.synchronize()
    if world > 1:
        dist.barrier()
    step_ms = [ev[i].elapsed_time(ev[i + 1]) for i in range(args.steps)]
    total_ms = ev[0].elapsed_time(ev[-1])
    status = run.sync_status()
    if status != native.TSS_OK:
        raise RuntimeError(f"device status {status} in the timed region")
    total_ms = max_over_ranks(total_ms, "cuda")
    ms = total_ms / args.steps
    value = job_tokens_per_s(w.n_rows, args.steps, world, total_ms)
    print(f"[bench] {w.name}: {ms * 1e3:.1f} us/step, {value:.1f} tokens/s", file=sys.stderr)

    # ---------------- e2e: host buffers through the C ABI, one sync per step ----------------
    e2e = None
    if not args.no_e2e:
        hres = run.alloc_results(len(w.requests), w.n_rows, logits=False, host=True)
        htoks = [torch.tensor(token_sets[v], dtype=torch.int32).pin_memory() for v in range(n_var)]
        hprobs = probs.cpu().pin_memory() if sample_mode else None
        hb = [run.batch(w.requests, tokens=htoks[v], io_host=True,
                        mode=native.TSS_MODE_SAMPLE if sample_mode else native.TSS_MODE_GREEDY,
                        temperature=w.temperature, draft_probs=hprobs, philox_seed=w.seed, philox_offset=v)
              for v in range(n_var)]
        for i in range(3):
            run.verify(hb[i % n_var], hres)
        torch.cuda.synchronize()
        n_e2e = max(10, min(args.steps, 100))
        acc_sum = 0
        t0 = time.perf_counter()
        for i in range(n_e2e):
            run.verify(hb[i % n_var], hres)
            stream.synchronize()
            acc_sum += int(hres["accept_len"].sum())
        e2e_s = time.perf_counter() - t0
        mean_accept = acc_sum / (n_e2e * len(w.requests))
        e2e = {"value": world * w.n_rows * n_e2e / e2e_s, "unit": "tokens/s",
               "h2d_bytes_per_step": STEP_DESC_BYTES + 4 * w.n_rows + (hprobs.numel() * 4 if sample_mode else 0),
               "d2h_bytes_per_step": 4 * (3 * len(w.requests) + hres["path"].numel()),
               "ms_per_step": e2e_s / n_e2e * 1e3, "steps": n_e2e,
               "copies": "per step: the step descriptor and the draft tokens (and draft probabilities when sampling) "
                         "host to device; accept_len, bonus, new_ctx_len and path device to host",
               "committed_tokens_per_s": world * len(w.requests) * (1 + mean_accept) * n_e2e / e2e_s,
               "mean_accept_len": mean_accept}

    # ---------------- per-kernel device times (CUDA events around every launch) ----------------
    roofline = None
    kernels = None
    peak, peak_kind = measured_peak()
    launches_per_step = None
    if True:
        # with --no-profile one profiled step still counts the launches of a step
        times = native.TssKernelTimes()
        n_prof = 1 if args.no_profile else max(5, min(args.steps, 20))
        for i in range(n_prof):
            run.v.verify_profiled(batches[i % n_var], run.kv_struct, res["_struct"], times, stream.cuda_stream)
        kernels = {}
        for k, name in enumerate(native.KERNEL_KINDS):
            if times.launches[k]:
                avg = times.ms[k] / times.launches[k]
                kernels[name] = {"launches_per_step": times.launches[k] / n_prof, "ms_per_step": times.ms[k] / n_prof,
                                 "avg_launch_us": avg * 1e3}
        kb = kernel_bytes(w, {n: v["launches_per_step"] for n, v in kernels.items()})
        for name, v in kernels.items():
            if name in kb:
                v["bytes_per_step"] = kb[name]
                v["gbs"] = kb[name] / (v["ms_per_step"] * 1e-3) / 1e9
        launches_per_step = sum(v["launches_per_step"] for v in kernels.values())
        tot = sum(v["ms_per_step"] for v in kernels.values())
        for v in kernels.values():
            v["share"] = v["ms_per_step"] / tot
        dom = max((n for n in kernels if n in kb), key=lambda n: kernels[n]["ms_per_step"])
        ach = kernels[dom]["gbs"]
        if "attention" in kernels:
            kernels["attention"]["impl"] = ATTENTION_IMPL.get(run.v.attention_kernel(), "attention")
        impl = kernels[dom].get("impl", dom)
        roofline = {"kernel": impl, "bound": "hbm", "achieved": ach, "peak": peak, "unit": "GB/s",
                    "frac": ach / peak, "peak_source": f"{peak_kind} copy bandwidth",
                    "frac_of_nominal_8TBs": ach / NOMINAL_HBM_GBS,
                    "bytes_per_launch": kb[dom] / kernels[dom]["launches_per_step"], "traffic": None}
        tr = find_traffic(args.traffic, impl, w.name)
        if tr is not None:
            roofline["traffic"] = tr["traffic_bytes"]
            roofline["traffic_source"] = tr.get("source")
        if args.no_profile:
            kernels = None
            roofline = None

    ab = synth.algorithmic_bytes(w)
    step_gbs = ab["total"] / (ms * 1e-3) / 1e9
    out = {
        "metric": METRIC, "value": value, "unit": "tokens/s", "n_gpus": world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": ms, "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "bf16", "data": "synthetic (seeded random-init weights, synthetic KV)",
        "config": workload_config(w, args),
        "latency_us": {"mean": ms * 1e3, "median": statistics.median(step_ms) * 1e3,
                       "p10": sorted(step_ms)[len(step_ms) // 10] * 1e3, "p90": sorted(step_ms)[(9 * len(step_ms)) // 10] * 1e3},
        "committed_tokens_per_s": None,
        "step_roofline": {"bytes_per_step": ab["total"], "weights": ab["weights"], "kv_read": ab["kv_read"],
                          "achieved_gbs": step_gbs, "frac_of_measured": step_gbs / peak,
                          "frac_of_nominal_8TBs": step_gbs / NOMINAL_HBM_GBS},
        "roofline": roofline, "kernels": kernels, "e2e": e2e,
        "gpu_launches": int(round(launches_per_step * args.steps)),
        "gpu_launches_per_step": launches_per_step,
        "clocks": clk.summary(),
    }
    # committed tokens: the mean accept length over the e2e steps, which cycle through the same
    # draft variants as the timed steps (the device-timed loop does not read results back)
    if e2e is not None:
        out["committed_tokens_per_s"] = world * len(w.requests) * (1 + e2e["mean_accept_len"]) * args.steps / (
            total_ms / 1e3)
        out["mean_accept_len"] = e2e["mean_accept_len"]
    if sample is not None:
        n_s = 3
        secs = [sample.step_seconds(i) for i in range(n_s)]
        sec = statistics.median(secs)
        out["cpu_baseline"] = {"value": w.n_rows / sec, "unit": "tokens/s", "cores": cores(), "kind": "oracle",
                               "sample": sample.describe(n_s), "seconds_per_step": sec,
                               "measured": isinstance(sample, OracleStep)}
    run.close()
    if rank == 0:
        print(json.dumps(out))
    if world > 1:
        dist.destroy_process_group()


def sweep_workload(name, n_skip):
    """Workload of a sweep point: the KV-bound 7B workload (B=16, ctx 16384, k=8) or the 7B chain
    (B=1, ctx 1024, k=5), with the first n_skip layers of one seeded permutation of layers 1..31
    skipped (nested sets, so each point adds layers to the previous one's skip set)."""
    from paper_2609_26100_gb300 import synth
    if name == "7b_long":
        return synth.workload_7b_long(n_skip=n_skip)
    if name == "7b_chain":
        perm = synth.seeded_permutation(list(range(1, synth.LLAMA2_7B.n_layers)), synth.DEFAULT_SEED, "7b_long.perm")
        return synth.workload_7b_chain(mask_layers=sorted(perm[:n_skip]))
    raise ValueError(f"--sweep supports the 7b_long and 7b_chain workloads, not {name}")


SWEEP_METRIC = {
    "7b_long": "7B KV-bound verify latency vs active layers (B=16, ctx 16384, k=8)",
    "7b_chain": "7B chain verify latency vs active layers (B=1, ctx 1024, k=5): the verification cost C_d(S)",
}


def run_sweep(args):
    """Verify latency against the number of active layers (the verification cost of a skip set,
    the C_d term of the paper's search objective): the skip sets are nested prefixes of one seeded
    permutation, the weights and the context KV of every layer are generated once, and each point
    is timed with CUDA events.  Prints one JSON line: the points, the least-squares line (slope,
    intercept, R^2) and each point's bytes against the measured and nominal HBM peaks."""
    import torch
    from paper_2609_26100_gb300 import build as _build
    from paper_2609_26100_gb300 import native, synth
    from paper_2609_26100_gb300.runner import TssRunner
    torch.cuda.set_device(0)
    _build.build()
    counts = [int(x) for x in args.sweep.split(",")]
    name = args.workload if args.workload in SWEEP_METRIC else "7b_long"
    dense = sweep_workload(name, 0)
    run = TssRunner.for_workload(dense)
    stream = torch.cuda.current_stream()
    peak, _ = measured_peak()
    points = []
    for n in counts:
        w = sweep_workload(name, n)
        run.set_phi(w.phi)
        res = run.alloc_results(len(w.requests), w.n_rows, logits=False)
        b = run.batch(w.requests)
        for _ in range(max(2, args.warmup)):
            run.verify(b, res)
        if run.sync_status() != native.TSS_OK:
            raise RuntimeError(f"device status error at {n} skipped layers")
        ev = [torch.cuda.Event(enable_timing=True) for _ in range(args.steps + 1)]
        torch.cuda.synchronize()
        ev[0].record(stream)
        for i in range(args.steps):
            run.verify(b, res)
            ev[i + 1].record(stream)
        torch.cuda.synchronize()
        ms = ev[0].elapsed_time(ev[-1]) / args.steps
        ab = synth.algorithmic_bytes(w)
        gbs = ab["total"] / (ms * 1e-3) / 1e9
        points.append({"skipped": n, "active_layers": ab["active_union"], "us_per_step": ms * 1e3,
                       "bytes_per_step": ab["total"], "achieved_gbs": gbs, "frac_of_measured": gbs / peak,
                       "frac_of_nominal_8TBs": gbs / NOMINAL_HBM_GBS})
        print(f"[sweep] skipped {n:2d}: {ms * 1e3:9.1f} us/step, {gbs:7.1f} GB/s", file=sys.stderr)
    run.close()
    xs = [p_["active_layers"] for p_ in points]
    ys = [p_["us_per_step"] for p_ in points]
    n = len(xs)
    mx, my = sum(xs) / n, sum(ys) / n
    sxx = sum((x - mx) ** 2 for x in xs)
    slope = sum((x - mx) * (y - my) for x, y in zip(xs, ys)) / sxx if sxx > 0 else 0.0
    icpt = my - slope * mx
    ss_tot = sum((y - my) ** 2 for y in ys)
    ss_res = sum((y - (icpt + slope * x)) ** 2 for x, y in zip(xs, ys))
    r2 = 1.0 - ss_res / ss_tot if ss_tot > 0 else 1.0
    print(json.dumps({"metric": SWEEP_METRIC[name], "workload": name,
                      "unit": "us/step", "higher_is_better": False, "steps": args.steps, "points": points,
                      "fit": {"slope_us_per_layer": slope, "intercept_us": icpt, "r2": r2},
                      "data": "synthetic (seeded random-init weights, synthetic KV)"}))


def run_prefill(args):
    """Prompt prefill under the 7B chain workload's skip configuration: 4 requests of
    args.prefill tokens each appended to empty caches with tss_prefill, timed with CUDA events.
    The default path runs each request's prompt in chunks of up to 1024 tokens through
    tokens-tiled tcgen05 GEMMs and a causal tcgen05 attention (TSS_PREFILL=steps: chains of up to
    64 tokens as verification steps of 256 rows).  Prints one JSON line: prompt tokens per second
    and the tensor throughput of the projections (2 x active parameters per token, both bf16
    parts counted as executed) against the measured bf16 peak."""
    import torch
    from paper_2609_26100_gb300 import build as _build
    from paper_2609_26100_gb300 import native, synth
    from paper_2609_26100_gb300.runner import TssRunner
    torch.cuda.set_device(0)
    _build.build()
    w = synth.workload_7b_chain()
    if args.layers:  # a cut of the model (profiling): the first args.layers layers
        import dataclasses
        w.arch = dataclasses.replace(w.arch, n_layers=args.layers)
        w.phi = {d: m & ((1 << args.layers) - 1) for d, m in w.phi.items()}
    a = w.arch
    union = w.active_union()
    n_req, n_tok = 4, args.prefill
    weights = synth.make_weights(a, w.seed, device="cuda", layers=union)
    for l in range(a.n_layers):
        if weights["layers"][l] is None:
            weights["layers"][l] = {k: torch.zeros(sh, dtype=torch.bfloat16, device="cuda")
                                    for k, sh in synth.layer_shapes(a).items()}
    run = TssRunner(a, weights, n_slots=n_req, kv_cap=n_tok + 8, max_batch=n_req, max_rows=256, max_nodes=64,
                    kv_layers=union)
    del weights
    torch.cuda.empty_cache()
    run.set_phi(w.phi)
    prompts = [synth.uniform_ints(n_tok, a.vocab, w.seed, f"prefill.{b}").tolist() for b in range(n_req)]
    doms = [w.requests[0].domain] * n_req
    stream = torch.cuda.current_stream()
    for _ in range(max(1, args.warmup)):
        run.prefill(prompts, [0] * n_req, doms)
    if run.sync_status() != native.TSS_OK:
        raise RuntimeError("device status error in prefill")
    ev0, ev1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    torch.cuda.synchronize()
    ev0.record(stream)
    for _ in range(args.steps):
        run.prefill(prompts, [0] * n_req, doms)
    ev1.record(stream)
    torch.cuda.synchronize()
    ms = ev0.elapsed_time(ev1) / args.steps
    steps_mode = os.environ.get("TSS_PREFILL") == "steps"
    layer_params = 4 * a.d_model * a.d_model + 3 * a.d_model * a.d_mlp
    useful = 2.0 * layer_params * len(union) * n_req * n_tok  # projection FLOPs (bf16 x weights)
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            peak_tf, peak_src = float(json.load(f)["bf16_tflops"]), "measured"
    except Exception:
        peak_tf, peak_src = 1900.0, "fallback"
    executed_tf = 2 * useful / (ms / 1e3) / 1e12  # hi and lo activation parts
    path = (f"{-(-n_tok // 64)} verification steps of 256 rows" if steps_mode else
            f"chunks of up to 1024 tokens per request: tokens-tiled tcgen05 GEMMs + causal tcgen05 attention")
    out = {"metric": "prompt prefill tokens/s under the 7B chain skip set (4 requests)", "value":
           n_req * n_tok / (ms / 1e3), "unit": "tokens/s", "higher_is_better": True, "n_gpus": 1,
           "steps": args.steps, "warmup": args.warmup, "ms_per_prefill": ms, "dtype": "bf16",
           "data": "synthetic (seeded random-init weights, uniform random prompt ids)",
           "config": {"workload": f"7b_chain skip set, {n_req} requests x {n_tok} prompt tokens, {path}",
                      "active_layers": len(union)},
           "roofline": {"bound": "tensor", "achieved": executed_tf, "peak": peak_tf, "unit": "TFLOP/s",
                        "frac": executed_tf / peak_tf, "peak_source": f"{peak_src} bf16",
                        "note": "projection FLOPs of both bf16 activation parts; attention not counted"}}
    run.close()
    print(json.dumps(out))


def run_grouped(args):
    """Domain-grouped verification against the mixed step: the same batch verified as one mixed
    step (every request completes when the union of active layers has streamed) and as one step per
    skip set (tss_verify_grouped, fewest active layers first); CUDA events give each group's
    completion time.  Prints one JSON line: per-request completion times of both, their means, and
    each group's layer count and bytes."""
    import torch
    from paper_2609_26100_gb300 import build as _build
    from paper_2609_26100_gb300 import native, synth
    from paper_2609_26100_gb300.runner import TssRunner
    torch.cuda.set_device(0)
    _build.build()
    name = args.workload if args.workload != "7b_chain" else "13b_mixed"
    w = make_workload(name, args.skip)
    run = TssRunner.for_workload(w)
    stream = torch.cuda.current_stream()
    sample = w.mode == "sample"
    kw = {}
    if sample:
        kw = dict(mode=native.TSS_MODE_SAMPLE, temperature=w.temperature,
                  draft_probs=torch.cat([r.draft_probs for r in w.requests], 0).cuda(), philox_seed=w.seed)
    B = len(w.requests)
    b = run.batch(w.requests, **kw)
    res = run.alloc_results(B, w.n_rows, logits=False)
    for _ in range(max(2, args.warmup)):
        run.verify(b, res)
        run.verify_grouped(b, res)
    if run.sync_status() != native.TSS_OK:
        raise RuntimeError("device status error")
    steps = max(3, min(args.steps, 50))
    mixed_ms, group_ms = [], []
    n_groups = 0
    for _ in range(steps):
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        run.verify(b, res)
        e1.record(stream)
        ev = [torch.cuda.Event(enable_timing=True) for _ in range(B)]
        g0 = torch.cuda.Event(enable_timing=True)
        g0.record(stream)
        n_groups = run.verify_grouped(b, res, events=ev)
        torch.cuda.synchronize()
        mixed_ms.append(e0.elapsed_time(e1))
        group_ms.append([g0.elapsed_time(ev[g]) for g in range(n_groups)])
    if run.sync_status() != native.TSS_OK:
        raise RuntimeError("device status error in the timed region")
    mixed = statistics.median(mixed_ms)
    gdone = [statistics.median(x[g] for x in group_ms) for g in range(n_groups)]
    # group of each request: skip sets ordered as the library orders them
    masks = [w.skip_mask(i) for i in range(B)]
    order = []
    for m in masks:
        if m not in order:
            order.append(m)
    order.sort(key=lambda m: w.arch.n_layers - bin(m).count("1"))
    per_req = [gdone[order.index(m)] for m in masks]
    groups = []
    for g, m in enumerate(order):
        members = [i for i in range(B) if masks[i] == m]
        ab = native.estimate_step_bytes(w.arch, [m] * len(members), [w.requests[i].ctx_len for i in members],
                                        [len(w.requests[i].parents) for i in members])
        groups.append({"skip": synth.layers_of(m), "requests": members, "active_layers": ab["active_union"],
                       "bytes": ab["total"], "done_us": gdone[g] * 1e3})
    run.close()
    print(json.dumps({
        "metric": "per-request completion time: mixed step vs domain-grouped steps", "workload": w.name,
        "unit": "us", "steps": steps, "mixed_step_us": mixed * 1e3,
        "grouped_total_us": gdone[-1] * 1e3, "grouped_request_us": [x * 1e3 for x in per_req],
        "mixed_request_mean_us": mixed * 1e3, "grouped_request_mean_us": statistics.mean(per_req) * 1e3,
        "requests_sooner_than_mixed": sum(1 for x in per_req if x < mixed), "groups": groups,
        "data": "synthetic (seeded random-init weights, synthetic KV)"}))


def main():
    args = parse_args()
    if args.impl == "reference":
        run_reference(args)
    elif args.sweep:
        run_sweep(args)
    elif args.prefill:
        run_prefill(args)
    elif args.grouped:
        run_grouped(args)
    else:
        run_tss(args)


if __name__ == "__main__":
    main()
