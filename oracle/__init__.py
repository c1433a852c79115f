"""CPU oracle for TSS target-side verification.

TEST INFRASTRUCTURE ONLY: a plain NumPy restatement of the paper's verifier (layer-skip
controller, LLaMA blocks, greedy and speculative-sampling acceptance, KV compaction) and of the
Philox4x32-10 generator.  Only tests/, __graft_entry__.smoke() and bench.py's cpu_baseline leg
may import it.  It shares no code with the CUDA library and imports nothing from it.
"""
from . import philox, tss_oracle  # noqa: F401
