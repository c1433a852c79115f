"""Where the persistent kernel's shared-memory plan fits (tss_persistent_plan, host arithmetic, no
GPU).  tss_verify runs a step only when it fits and otherwise returns UNSUPPORTED_ARCH (there is
no silent fallback), so these tests map the whole range of row counts at the 7B and 13B widths."""
import pytest

from paper_2609_26100_gb300 import native, synth

SMS = 152  # GB300
SMEM_LIMIT = 232448  # per-block dynamic shared memory of sm_103 (227 KiB)


@pytest.mark.parametrize("arch", [synth.LLAMA2_7B, synth.LLAMA2_13B], ids=["7b", "13b"])
def test_plan_fits_every_row_count(arch):
    """Every batch shape the context limits allow (1..64 requests, up to 256 rows, up to 64 nodes a
    request) fits, at short (the chain and tree workloads) and long (16k) contexts."""
    seen = set()
    for M in range(1, 257):
        for B in sorted({1, (M + 127) // 128, (M + 63) // 64, min(M, 8), min(M, 16), min(M, 64)}):
            if B < (M + 127) // 128 or B > M:
                continue
            for keys in (1, 1030, 2109, 4101, 16393):
                plan = native.persistent_plan(arch, B, M, keys, SMS)
                assert plan["fits"], (M, B, keys)
                assert plan["smem_bytes"] <= SMEM_LIMIT
                assert plan["stages"] >= 2 and 1 <= plan["kps"] <= 3
                seen.add((plan["kps"], plan["stages"]))
    assert len(seen) > 1  # the ring shrinks as the B operand grows


def test_plan_of_the_benchmark_steps():
    """The plans the benchmark workloads run with: 48 KiB weight stages for the 7B chain."""
    chain = native.persistent_plan(synth.LLAMA2_7B, 1, 6, 1030, SMS)
    assert chain["fits"] and chain["kps"] == 3 and chain["stages"] == 3
    tree = native.persistent_plan(synth.LLAMA2_7B, 1, 61, 2109, SMS)
    assert tree["fits"]
    mixed = native.persistent_plan(synth.LLAMA2_13B, 8, 48, 4101, SMS)
    assert mixed["fits"]
    wide = native.persistent_plan(synth.LLAMA2_7B, 2, 228, 2109, SMS)
    assert wide["fits"]


def test_plan_rejects_bad_arguments():
    for args in [(0, 6, 10, SMS), (65, 100, 10, SMS), (1, 257, 10, SMS), (2, 1, 10, SMS), (1, 6, 0, SMS),
                 (1, 6, 10, 0)]:
        with pytest.raises(native.TssError) as err:
            native.persistent_plan(synth.LLAMA2_7B, *args)
        assert err.value.status == native.TSS_ERR_INVALID_ARG
