"""bench.py's own launch of N replicas (`--gpus N` without a launcher) on the
CPU: two `gloo` ranks started by bench.spawn_replicas under
torch.distributed.run, each timing its replica with bench.time_replicas
(barrier and synchronisation on both sides, max over ranks), and the job's
fields from bench.replica_fields.  The rank program's step only sleeps."""
import json
import os
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)

import bench  # noqa: E402

RANK_PROGRAM = os.path.join(os.path.dirname(os.path.abspath(__file__)), "bench_replica_rank.py")


def test_spawned_replicas_report_job_value(tmp_path):
    steps, ops = 3, 2.0e12
    rc = bench.spawn_replicas(2, [RANK_PROGRAM, str(tmp_path), str(steps), str(ops)])
    assert rc == 0
    ranks = [json.load(open(tmp_path / f"rank{r}.json")) for r in range(2)]
    assert [r["rank"] for r in ranks] == [0, 1] and all(r["world"] == 2 for r in ranks)
    # rank 1 sleeps twice as long per step: it is the slowest, and every
    # rank agrees on the job's time
    assert ranks[1]["ms"] > ranks[0]["ms"]
    job_ms = max(r["ms"] for r in ranks)
    assert all(r["job_ms"] == pytest.approx(job_ms) for r in ranks)
    assert ranks[1]["ms"] >= steps * 40
    job = json.load(open(tmp_path / "job.json"))
    assert job["n_gpus"] == 2 and job["scaling"] == "weak"
    assert job["parallelism"] == "replicas x2"
    # the work of both ranks over the slowest rank's time
    assert job["value"] == pytest.approx(2 * steps * ops / (job_ms * 1e-3) / 1e12)
    assert job["ms_per_step"] == pytest.approx(job_ms / steps)


def test_gpu_arm_refuses_more_replicas_than_devices(monkeypatch):
    # on a machine without N visible GPUs the launch stops with a message
    # instead of starting ranks that would share one device
    monkeypatch.delenv("WORLD_SIZE", raising=False)
    monkeypatch.setattr(sys, "argv", ["bench.py", "--gpus", "64"])
    with pytest.raises(SystemExit) as exc:
        bench.main()
    assert "64" in str(exc.value)


def test_one_replica_fields():
    f = bench.replica_fields(1, 1.0e12, 2, 500.0)
    assert f["n_gpus"] == 1 and f["parallelism"] == "1 GPU"
    assert f["value"] == pytest.approx(4.0)
