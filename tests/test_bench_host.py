"""The benchmark's reference arm on the CPU: its JSON line keeps the contract
(the same config as the GPU arm's, the oracle as its CPU baseline, no host
copies), and under a multi-rank launch only rank 0 prints."""
import json
import os
import subprocess
import sys

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _run(env_extra, *args):
    env = dict(os.environ, **env_extra)
    env.pop("CUDA_VISIBLE_DEVICES", None)
    return subprocess.run([sys.executable, os.path.join(ROOT, "bench.py"), *args],
                          cwd=ROOT, env=env, capture_output=True, text=True, timeout=300)


def test_reference_arm_line():
    res = _run({}, "--impl", "reference", "--workload", "tiny", "--steps", "1", "--warmup", "3")
    assert res.returncode == 0, res.stderr
    lines = [ln for ln in res.stdout.splitlines() if ln.startswith("{")]
    assert len(lines) == 1
    d = json.loads(lines[0])
    assert d["impl"] == "reference"
    assert d["metric"] == "candidate sets scored/sec" and d["unit"] == "sets/s"
    assert d["higher_is_better"] is True and d["steps"] == 1 and d["warmup"] >= 3
    assert d["value"] > 0 and d["cpu_baseline"]["value"] == d["value"]
    assert d["cpu_baseline"]["kind"] == "oracle" and d["cpu_baseline"]["cores"] >= 1
    assert d["e2e"]["value"] == d["value"]
    assert d["e2e"]["h2d_bytes_per_step"] == 0 and d["e2e"]["d2h_bytes_per_step"] == 0
    cfg = d["config"]
    # the GPU arm's config keys: the workload and its sizes
    for k in ("workload", "R", "N", "T", "C", "total_prefix", "Hq", "Hkv", "d", "D", "V", "Hl",
              "parallelism", "lm_head", "recurrence", "l2"):
        assert k in cfg, k
    assert cfg["workload"] == "tiny" and cfg["R"] == 1 and cfg["N"] == 7 and cfg["T"] == 10


def test_reference_arm_is_silent_on_other_ranks():
    res = _run({"RANK": "1", "LOCAL_RANK": "1", "WORLD_SIZE": "2"}, "--impl", "reference",
               "--workload", "tiny", "--steps", "1", "--warmup", "3")
    assert res.returncode == 0, res.stderr
    assert not [ln for ln in res.stdout.splitlines() if ln.startswith("{")]
