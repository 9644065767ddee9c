"""The bench's reference arm on CPU: `bench.py --impl reference` times the
oracle and prints one JSON line with the contract's keys; under torchrun only
rank 0 does so, the other ranks exit 0 without work."""
import json
import os
import sys

import pytest

sys.path.insert(0, os.path.dirname(os.path.dirname(os.path.abspath(__file__))))
import bench  # noqa: E402


def _last_json(text):
    lines = [ln for ln in text.strip().splitlines() if ln.startswith("{")]
    assert lines, text
    return json.loads(lines[-1])


def test_reference_arm_prints_the_contract_line(capsys, monkeypatch):
    for v in ("RANK", "WORLD_SIZE", "LOCAL_RANK"):
        monkeypatch.delenv(v, raising=False)
    assert bench.main(["--impl", "reference", "--config", "tiny", "--steps", "2", "--warmup", "3"]) == 0
    d = _last_json(capsys.readouterr().out)
    for key in ("metric", "value", "unit", "n_gpus", "steps", "warmup", "ms_per_step", "higher_is_better",
                "scaling", "vs_baseline", "dtype", "data", "config", "cpu_baseline", "e2e"):
        assert key in d, key
    assert d["impl"] == "reference"
    assert d["steps"] == 2 and d["warmup"] == 3 and d["n_gpus"] == 1
    assert d["value"] > 0 and d["ms_per_step"] > 0 and d["higher_is_better"] is True
    assert d["config"]["workload"].startswith("tiny")
    cb = d["cpu_baseline"]
    assert cb["kind"] == "oracle" and cb["cores"] >= 1 and cb["sample"] and cb["value"] == d["value"]
    e = d["e2e"]
    assert e["value"] == d["value"] and e["unit"] == d["unit"]
    assert e["h2d_bytes_per_step"] == 0 and e["d2h_bytes_per_step"] == 0


def test_reference_arm_on_a_nonroot_rank_is_silent(capsys, monkeypatch):
    monkeypatch.setenv("RANK", "1")
    monkeypatch.setenv("WORLD_SIZE", "2")
    monkeypatch.setenv("LOCAL_RANK", "1")
    assert bench.main(["--impl", "reference", "--config", "tiny", "--steps", "1", "--warmup", "3",
                       "--gpus", "2"]) == 0
    assert capsys.readouterr().out.strip() == ""


def test_warmup_below_three_is_refused():
    with pytest.raises(SystemExit):
        bench.main(["--impl", "reference", "--config", "tiny", "--steps", "1", "--warmup", "2"])
