"""bench.py's launch contract on CPU: `--gpus N` really starts N ranks (here
with gloo, no kernels), a launcher whose rank count differs from --gpus is
refused, and the reference arm reports the time it measured on its sample
(with the same config as the GPU arm), not a projection."""
import json
import os
import subprocess
import sys

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _run(args, env=None, timeout=300):
    e = dict(os.environ)
    e.pop("WORLD_SIZE", None)
    e.pop("RANK", None)
    e.pop("LOCAL_RANK", None)
    e["CUDA_VISIBLE_DEVICES"] = ""
    e.update(env or {})
    return subprocess.run([sys.executable, os.path.join(ROOT, "bench.py")] + args, cwd=ROOT, env=e,
                          capture_output=True, text=True, timeout=timeout)


def _json_lines(out):
    return [json.loads(ln) for ln in out.splitlines() if ln.startswith("{")]


def test_gpus_2_starts_two_ranks():
    r = _run(["--gpus", "2", "--launch-check"])
    assert r.returncode == 0, r.stderr[-2000:]
    lines = _json_lines(r.stdout)
    assert len(lines) == 1                      # rank 0 alone prints
    assert lines[0]["world"] == 2 and lines[0]["ranks_seen"] == 2


def test_rank_count_mismatch_is_refused():
    r = _run(["--gpus", "4", "--launch-check"], env={"WORLD_SIZE": "1", "RANK": "0", "LOCAL_RANK": "0"})
    assert r.returncode != 0
    assert "--gpus 4" in r.stderr


def test_reference_arm_reports_its_measured_step():
    r = _run(["--impl", "reference", "--steps", "2", "--warmup", "0", "--ref-rows", "2"], timeout=600)
    assert r.returncode == 0, r.stderr[-2000:]
    (line,) = _json_lines(r.stdout)
    assert line["impl"] == "reference" and line["sample_tokens_per_step"] == 2
    # the step time is the measured one: 2 steps of a 2-token sample take seconds, not minutes
    assert 0 < line["ms_per_step"] < 60_000
    import bench
    assert line["config"] == bench.workload_config(1)
    assert line["e2e"]["h2d_bytes_per_step"] == 0
