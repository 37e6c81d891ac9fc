"""The reference arm's JSON line (bench.py --impl reference): the oracle timed on host cores, in
the same metric and unit as the GPU arm, with the keys the harness reads. The oracle sample itself
(a 7B-shaped model in fp64) is replaced by a stub here; what is checked is the line's shape."""
import json

import bench


def test_reference_line_has_the_contract_keys(monkeypatch, capsys):
    sample = dict(value=0.5, unit="tokens/s", cores=4, kind="oracle", sample="stub sample", dtype="f64",
                  ms_per_iteration=6000.0, tokens_per_iteration=3.0, iterations=3)
    seen = []
    monkeypatch.setattr(bench, "oracle_sample", lambda steps, warmup, prompt_len: seen.append(
        (steps, warmup, prompt_len)) or (sample, None))

    class Args:
        steps, warmup, gpus, cpu_baseline_prompt = 3, 1, 1, 16

    bench.run_reference(Args, rank=0)
    line = json.loads(capsys.readouterr().out.strip().splitlines()[-1])
    assert line["impl"] == "reference" and line["metric"] == bench.METRIC
    assert line["value"] == 0.5 and line["unit"] == "tokens/s" and line["higher_is_better"] is True
    assert line["cpu_baseline"]["kind"] == "oracle" and line["cpu_baseline"]["cores"] == 4
    assert line["e2e"] == {"value": 0.5, "unit": "tokens/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}
    assert line["config"]["workload"] == bench.DEFAULT_WORKLOAD
    # one step = one oracle iteration: K timed after W untimed
    assert seen == [(3, 1, 16)] and line["ms_per_step"] == 6000.0 and line["dtype"] == "f64"
    for k in ("n_gpus", "steps", "warmup", "ms_per_step", "scaling", "vs_baseline", "dtype", "data"):
        assert k in line


def test_reference_arm_prints_unavailable_when_the_host_is_too_small(monkeypatch, capsys):
    monkeypatch.setattr(bench, "oracle_sample", lambda steps, warmup, prompt_len: (None, "host memory 8 GiB < 70 GiB needed"))

    class Args:
        steps, warmup, gpus, cpu_baseline_prompt = 3, 1, 1, 16

    bench.run_reference(Args, rank=0)
    line = json.loads(capsys.readouterr().out.strip())
    assert line == {"impl": "reference", "unavailable": "host memory 8 GiB < 70 GiB needed"}


def test_reference_arm_is_rank_zero_only(monkeypatch, capsys):
    monkeypatch.setattr(bench, "oracle_sample", lambda steps, warmup, prompt_len: (_ for _ in ()).throw(AssertionError))

    class Args:
        steps, warmup, gpus, cpu_baseline_prompt = 3, 1, 2, 16

    bench.run_reference(Args, rank=1)
    assert capsys.readouterr().out == ""
