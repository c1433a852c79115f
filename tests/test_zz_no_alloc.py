"""tss_linear_static, the allocation-free linear layer, for callers that cannot allocate device
memory when they run it (a plugin inside a framework that owns the device memory pool, a fixed
memory budget, or a loop that must not call cudaMalloc/cudaFree).  It keeps its stream-K scratch
in a static device array; this test checks it against tss_linear (the context-owning entry point)
through the C ABI on two calls in a row, so a second call sees the scratch the first one left.
The file is collected last."""
import numpy as np
import pytest
import torch

from paper_2609_26100_gb300 import native, synth

pytestmark = pytest.mark.gpu


def test_static_linear_matches_linear_on_two_calls():
    from paper_2609_26100_gb300 import build
    build.build()
    arch = synth.TINY
    w = synth.make_weights(arch, device="cuda")
    ref_ctx = native.Verifier(w, arch, max_batch=1, max_rows=64)
    try:
        for m, k, n in [(6, 4096, 1024), (13, 512, 384), (64, 256, 256)]:
            x = synth.normal_bf16((m, k), 7, f"nx{m}", 1.0).cuda()
            wt = synth.normal_bf16((n, k), 7, f"nw{n}", 0.05).cuda()
            y_ref = torch.empty((m, n), dtype=torch.float32, device="cuda")
            ref_ctx.linear(x, wt, y_ref)
            for call in range(2):
                y = torch.full((m, n), float("nan"), dtype=torch.float32, device="cuda")
                native.linear_static(x, wt, y)
                torch.cuda.synchronize()
                np.testing.assert_allclose(y.cpu().numpy(), y_ref.cpu().numpy(), rtol=1e-4, atol=1e-4,
                                           err_msg=f"{m}x{k}x{n} call {call}")
        # beyond the stated limits: a clear error, nothing launched
        x = torch.zeros((65, 64), dtype=torch.bfloat16, device="cuda")
        wt = torch.zeros((128, 64), dtype=torch.bfloat16, device="cuda")
        y = torch.zeros((65, 128), dtype=torch.float32, device="cuda")
        with pytest.raises(native.TssError) as err:
            native.linear_static(x, wt, y)
        assert err.value.status == native.TSS_ERR_INVALID_ARG
    finally:
        ref_ctx.close()
