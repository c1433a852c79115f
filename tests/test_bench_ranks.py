"""Host logic of bench.py's multi-process (one replica per GPU) mode, on CPU with gloo:
max-over-ranks timing, the whole-job value, and the reference arm running on rank 0 only."""
import json
import os
import socket
import sys

import pytest
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)
import bench  # noqa: E402


def _free_port():
    s = socket.socket()
    s.bind(("127.0.0.1", 0))
    port = s.getsockname()[1]
    s.close()
    return port


def _rank_main(rank, world, port, out_dir):
    import torch.distributed as dist
    dist.init_process_group("gloo", init_method=f"tcp://127.0.0.1:{port}", rank=rank, world_size=world)
    local_ms = 10.0 * (rank + 1)  # rank 1 is the slower replica
    job_ms = bench.max_over_ranks(local_ms, "cpu")
    value = bench.job_tokens_per_s(6, 4, world, job_ms)
    with open(os.path.join(out_dir, f"rank{rank}.json"), "w") as f:
        json.dump({"job_ms": job_ms, "value": value}, f)
    dist.destroy_process_group()


def test_two_replicas_take_the_slowest_rank(tmp_path):
    world, port = 2, _free_port()
    mp.spawn(_rank_main, args=(world, port, str(tmp_path)), nprocs=world, join=True)
    res = [json.load(open(tmp_path / f"rank{r}.json")) for r in range(world)]
    for r in res:
        assert r["job_ms"] == 20.0  # the max over ranks, on every rank
        assert r["value"] == pytest.approx(2 * 6 * 4 / 0.020)  # whole-job rows per second


def test_single_process_time_is_its_own():
    assert bench.max_over_ranks(7.5, "cpu") == 7.5
    assert bench.job_tokens_per_s(6, 10, 1, 5.0) == pytest.approx(6 * 10 / 0.005)


def test_reference_arm_runs_on_rank_zero_only(monkeypatch, capsys):
    monkeypatch.setenv("RANK", "1")
    monkeypatch.setattr(sys, "argv", ["bench.py", "--impl", "reference", "--workload", "tiny", "--steps", "1",
                                      "--warmup", "0"])
    args = bench.parse_args()
    bench.run_reference(args)
    assert capsys.readouterr().out == ""


def test_traffic_record_needs_same_kernel_workload_and_sources(tmp_path):
    rec = {"kernel": "attention", "workload": "7b_long", "traffic_bytes": 123,
           "sources_sha256": bench.kernel_sources_hash("attention")}
    (tmp_path / "a_traffic.txt").write_text(json.dumps(rec))
    assert bench.find_traffic(str(tmp_path), "attention", "7b_long")["traffic_bytes"] == 123
    assert bench.find_traffic(str(tmp_path / "a_traffic.txt"), "attention", "7b_long") is not None
    assert bench.find_traffic(str(tmp_path), "attention", "13b_mixed") is None
    assert bench.find_traffic(str(tmp_path), "verify_persistent", "7b_long") is None
    (tmp_path / "a_traffic.txt").write_text(json.dumps(dict(rec, sources_sha256="0" * 64)))
    assert bench.find_traffic(str(tmp_path), "attention", "7b_long") is None  # kernel changed since
    # the hash ignores comments and blank lines but not code
    assert bench.kernel_sources_hash("attention") != bench.kernel_sources_hash("verify_persistent")
