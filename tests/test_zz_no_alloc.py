"""tss_linear_static, the allocation-free linear layer, for callers that cannot allocate device
memory when they run it (a plugin inside a framework that owns the device memory pool, a fixed
memory budget, or a loop that must not call cudaMalloc/cudaFree).  It keeps its stream-K scratch
and status word in static device arrays.  Through the C ABI, on two calls in a row (so that the
second call sees the scratch the first one left), the result is checked against tss_linear (the
context-owning entry point) and against the product of x and w in float64; the device's free
memory does not change after the first call; the scratch bound is exact.  The file is collected
last."""
import numpy as np
import pytest
import torch

from paper_2609_26100_gb300 import native, synth

pytestmark = pytest.mark.gpu

SCRATCH_BYTES = 8 << 20


def _ref(x, wt):
    return x.double().cpu().numpy() @ wt.double().cpu().numpy().T


def test_static_linear_matches_linear_and_float64_on_two_calls():
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
            exact = _ref(x, wt)
            for call in range(2):
                y = torch.full((m, n), float("nan"), dtype=torch.float32, device="cuda")
                native.linear_static(x, wt, y)
                assert native.linear_static_status() == native.TSS_OK
                got = y.cpu().numpy()
                np.testing.assert_allclose(got, y_ref.cpu().numpy(), rtol=1e-4, atol=1e-4,
                                           err_msg=f"{m}x{k}x{n} call {call} vs tss_linear")
                np.testing.assert_allclose(got, exact, rtol=1e-4, atol=1e-4, err_msg=f"{m}x{k}x{n} call {call} vs fp64")
        # beyond the stated row limit: a clear error, nothing launched
        x = torch.zeros((65, 64), dtype=torch.bfloat16, device="cuda")
        wt = torch.zeros((128, 64), dtype=torch.bfloat16, device="cuda")
        y = torch.zeros((65, 128), dtype=torch.float32, device="cuda")
        with pytest.raises(native.TssError) as err:
            native.linear_static(x, wt, y)
        assert err.value.status == native.TSS_ERR_INVALID_ARG
    finally:
        ref_ctx.close()


def test_static_linear_at_the_scratch_limit_and_no_memory_change():
    """64 rows: the largest n_out whose stream-K scratch fits the 8 MiB array runs and is exact;
    one more tile of 128 outputs is rejected.  After the first call (which loads the module and
    reserves the array) later calls leave the device's free memory unchanged."""
    from paper_2609_26100_gb300 import build
    build.build()
    sms = torch.cuda.get_device_properties(0).multi_processor_count
    m, k = 64, 256
    tiles = SCRATCH_BYTES // (128 * m * 4) - sms  # (grid + tiles) * 128 * 64 rows * 4 bytes <= 8 MiB
    assert tiles * (k // 64) >= sms  # one CTA per SM: the grid is the SM count
    x = synth.normal_bf16((m, k), 9, "lim.x", 1.0).cuda()
    wt = synth.normal_bf16((tiles * 128, k), 9, "lim.w", 0.05).cuda()
    y = torch.empty((m, tiles * 128), dtype=torch.float32, device="cuda")
    native.linear_static(x, wt, y)
    assert native.linear_static_status() == native.TSS_OK
    free0 = torch.cuda.mem_get_info()[0]
    for _ in range(2):
        y.fill_(float("nan"))
        native.linear_static(x, wt, y)
        assert native.linear_static_status() == native.TSS_OK
    assert torch.cuda.mem_get_info()[0] == free0
    np.testing.assert_allclose(y.cpu().numpy(), _ref(x, wt), rtol=1e-4, atol=1e-4)
    wt2 = torch.zeros(((tiles + 1) * 128, k), dtype=torch.bfloat16, device="cuda")
    y2 = torch.zeros((m, (tiles + 1) * 128), dtype=torch.float32, device="cuda")
    with pytest.raises(native.TssError) as err:
        native.linear_static(x, wt2, y2)
    assert err.value.status == native.TSS_ERR_INVALID_ARG
    assert "8 MiB" in str(err.value)
