"""bench.py on the host: the reference arm's JSON line and the workload labels.

The reference arm times the fp64 oracle on the host cores, so it runs here
without a GPU. Its line must carry the keys of the bench line contract, with
`impl: reference` and a zero-byte `e2e`; under torchrun only rank 0 prints.
"""
import json
import os
import subprocess
import sys

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)

import bench  # noqa: E402
from synth import CONFIGS  # noqa: E402


def _run(extra_env=None):
    env = dict(os.environ)
    env.update(extra_env or {})
    r = subprocess.run([sys.executable, os.path.join(ROOT, "bench.py"), "--impl", "reference",
                        "--workload", "tiny", "--steps", "1", "--warmup", "0"],
                       capture_output=True, text=True, env=env, timeout=300)
    assert r.returncode == 0, r.stderr
    return [json.loads(x) for x in r.stdout.splitlines() if x.startswith("{")]


def test_reference_arm_prints_one_contract_line():
    lines = _run()
    assert len(lines) == 1
    d = lines[0]
    assert d["impl"] == "reference"
    for k in ("metric", "value", "unit", "n_gpus", "steps", "warmup", "ms_per_step",
              "higher_is_better", "scaling", "vs_baseline", "dtype", "data", "config"):
        assert k in d, k
    assert d["value"] > 0 and d["higher_is_better"] is True and d["steps"] == 1
    assert d["config"]["workload"].startswith("tiny:")
    cb = d["cpu_baseline"]
    assert cb["kind"] == "oracle" and cb["cores"] >= 1 and cb["value"] == d["value"] and cb["sample"]
    e2e = d["e2e"]
    assert e2e["value"] == d["value"] and e2e["unit"] == d["unit"]
    assert e2e["h2d_bytes_per_step"] == 0 and e2e["d2h_bytes_per_step"] == 0


def test_reference_arm_prints_nothing_on_other_ranks():
    assert _run({"RANK": "1", "WORLD_SIZE": "2", "LOCAL_RANK": "1"}) == []


def test_workload_labels_name_the_head_and_the_l2_case():
    head = bench.config_of(CONFIGS["llada8b_r512_onpolicy"])
    assert head["workload"].startswith("llada8b_r512_onpolicy: LLaDA-8B-shaped LM head H=4096 "
                                       "V=126464, 16 responses x (prompt 256 + response 512)")
    assert head["l2"].startswith("inputs larger than L2")
    dream = bench.config_of(CONFIGS["dream7b"])
    assert "Dream-7B-shaped LM head" in dream["workload"] and "1.09 GB" in dream["l2"]
    tiny = bench.config_of(CONFIGS["tiny"])
    assert "LLaDA" not in tiny["workload"] and tiny["l2"].startswith("inputs fit in L2")
