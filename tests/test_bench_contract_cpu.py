"""The bench line's shape on CPU: the reference arm (the fp64 oracle timed on the host cores) of
the default workload prints one JSON line with every key the bench contract names, so that the
driver can pair it with the GPU arm's line; and the GPU arm refuses to run without a GPU instead
of falling back to the CPU."""
import json

import pytest

CONTRACT_KEYS = {"metric", "value", "unit", "n_gpus", "steps", "warmup", "ms_per_step",
                 "higher_is_better", "scaling", "vs_baseline", "dtype", "data", "config"}


def _bench():
    import bench
    return bench


def test_reference_arm_line_keeps_the_contract(monkeypatch, capsys):
    b = _bench()
    for k in ("RANK", "WORLD_SIZE", "LOCAL_RANK"):
        monkeypatch.delenv(k, raising=False)

    class Args:
        steps, warmup = 2, 3

    w = b.workload("llama8b_layer_b8_s4096")
    b.run_reference(Args, w)
    lines = [ln for ln in capsys.readouterr().out.splitlines() if ln.startswith("{")]
    assert len(lines) == 1
    d = json.loads(lines[0])
    assert CONTRACT_KEYS <= set(d)
    assert d["impl"] == "reference"
    assert d["config"]["workload"] == "llama8b_layer_b8_s4096"
    assert d["unit"] == "macro-steps/s" and d["higher_is_better"] is True
    assert d["value"] > 0 and d["n_gpus"] == 1 and d["steps"] == 2 and d["warmup"] >= 3
    assert d["ms_per_step"] == pytest.approx(1e3 / d["value"], rel=1e-2)
    assert d["dtype"] == "f64" and d["data"] == "synthetic" and d["vs_baseline"] is None
    cb = d["cpu_baseline"]
    assert cb["kind"] == "oracle" and cb["value"] == d["value"] and cb["cores"] >= 1
    assert cb["sample"]
    e = d["e2e"]
    assert (e["value"], e["unit"]) == (d["value"], d["unit"])
    assert e["h2d_bytes_per_step"] == 0 and e["d2h_bytes_per_step"] == 0
    # the GPU arm's line names the same metric on the same workload
    assert d["metric"] == b.METRIC


def test_gpu_arm_does_not_fall_back_to_the_cpu(monkeypatch):
    import torch
    if torch.cuda.is_available():
        pytest.skip("a GPU is present")
    b = _bench()
    for k in ("RANK", "WORLD_SIZE", "LOCAL_RANK"):
        monkeypatch.delenv(k, raising=False)
    monkeypatch.setattr("sys.argv", ["bench.py", "--steps", "1", "--warmup", "3"])
    with pytest.raises(SystemExit) as e:
        b.main()
    assert "needs a GPU" in str(e.value.code)
