"""tss_estimate_step_bytes (host arithmetic of the C ABI, no GPU) against the byte count bench.py
uses for its roofline (synth.algorithmic_bytes, a separate Python implementation): the five
benchmark workloads, random mixed batches, and the argument checks."""
import dataclasses
import os

import numpy as np
import pytest

from paper_2609_26100_gb300 import native, synth

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _c_bytes(w):
    reqs = w.requests
    return native.estimate_step_bytes(w.arch, [w.skip_mask(b) for b in range(len(reqs))],
                                      [r.ctx_len for r in reqs], [len(r.parents) for r in reqs])


@pytest.mark.parametrize("make", [synth.workload_7b_chain, lambda: synth.workload_7b_chain(mask_layers=()),
                                  synth.workload_7b_tree, synth.workload_13b_mixed, synth.workload_7b_long])
def test_benchmark_workloads(make):
    w = make()
    got, want = _c_bytes(w), synth.algorithmic_bytes(w)
    for k in ("weights", "kv_read", "kv_write", "total", "active_union"):
        assert got[k] == want[k], k


def test_7b_chain_step_moves_12_07_gb():
    assert _c_bytes(synth.workload_7b_chain())["total"] == 12067667968


def test_random_mixed_batches():
    rng = np.random.default_rng(0)
    for trial in range(50):
        L = int(rng.integers(1, 65))
        arch = dataclasses.replace(synth.TINY, n_layers=L, d_model=128 * int(rng.integers(1, 5)),
                                   d_mlp=8 * int(rng.integers(1, 100)), vocab=int(rng.integers(1, 5000)))
        B = int(rng.integers(1, 9))
        phi = {d: int(sum(1 << l for l in range(L) if rng.random() < 0.3)) for d in range(B)}
        ctx = [int(x) for x in rng.integers(0, 5000, B)]
        w = synth.config_chain(arch, f"rand{trial}", B, ctx, int(rng.integers(0, 9)), phi, list(range(B)), 1)
        got, want = _c_bytes(w), synth.algorithmic_bytes(w)
        assert got == {k: want[k] for k in got}


def test_skipping_a_layer_saves_its_weights_and_kv():
    a = synth.LLAMA2_7B
    dense = native.estimate_step_bytes(a, [0], [1024], [6])
    one = native.estimate_step_bytes(a, [1 << 5], [1024], [6])
    assert dense["weights"] - one["weights"] == a.layer_weight_bytes == 404750336
    assert dense["kv_read"] - one["kv_read"] == 1024 * a.kv_bytes_per_token
    assert one["active_union"] == 31


def test_argument_checks():
    a = synth.TINY
    with pytest.raises(native.TssError) as e:
        native.estimate_step_bytes(a, [1 << a.n_layers], [0], [1])
    assert e.value.status == native.TSS_ERR_INVALID_ARG
    with pytest.raises(native.TssError):
        native.estimate_step_bytes(a, [0], [-1], [1])
    with pytest.raises(native.TssError):
        native.estimate_step_bytes(a, [], [], [])


def test_bench_counts_the_step_descriptor_it_uploads(tmp_path):
    """bench.py's e2e copy count includes the per-step descriptor: its constant equals the size of
    the struct tss_verify copies (compiled here with nvcc, host code only)."""
    import shutil
    import subprocess
    import bench
    nvcc = shutil.which("nvcc") or "/usr/local/cuda/bin/nvcc"
    if not os.path.exists(nvcc) and not shutil.which("nvcc"):
        pytest.skip("no nvcc")
    src = tmp_path / "sd.cu"
    src.write_text('#include "common.cuh"\n#include <cstdio>\n'
                   'int main() { printf("%zu\\n", sizeof(tss::StepDesc)); return 0; }\n')
    exe = tmp_path / "sd"
    csrc = os.path.join(ROOT, "paper_2609_26100_gb300", "csrc")
    r = subprocess.run([nvcc, "-std=c++17", "-I", csrc, str(src), "-o", str(exe)], capture_output=True, text=True)
    assert r.returncode == 0, r.stderr
    out = subprocess.run([str(exe)], capture_output=True, text=True, check=True).stdout
    assert int(out) == bench.STEP_DESC_BYTES
