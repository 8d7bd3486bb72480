"""Host logic of bench.py on CPU: the default arguments the run contract needs,
the algorithmic bytes of a step (the roofline's numerator), the rule that a
committed ncu summary feeds `traffic` only when it was taken on the current
row-pass source (and, with filters, at the same top-k), the reference
arm's JSON line (the oracle on the host cores) and the count of DTW band
cells behind the band-cells-per-second figure."""
import json
import os
import subprocess
import sys
from types import SimpleNamespace

import numpy as np
import pytest
import torch

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)
import bench  # noqa: E402


def test_defaults_are_one_gpu_and_enough_warmup():
    a = bench.parse_args([])
    assert a.gpus == 1 and a.impl == "mine" and a.warmup >= 3
    assert a.workload == bench.DEFAULT_WORKLOAD
    assert a.top_k == 0 and a.top_p == 1.0 and a.shards == 0


def test_algorithmic_bytes_count_each_distinct_mapped_draft_row_once():
    # request 0: targets map to draft rows 0, 0, 2 (two distinct rows, 3 target
    # rows + its bonus row); request 1: one target mapped to row 1 (one distinct
    # row, 1 target row + bonus)
    wl = SimpleNamespace(
        B=2, n_target=4, target_off=np.array([0, 3, 4]),
        draft_logits=torch.empty(5, 100, dtype=torch.float32),
        target_logits=torch.empty(6, 300, dtype=torch.bfloat16))
    mp = np.array([0, 0, 2, 1])
    ab = bench.algorithmic_bytes(wl, mp)
    assert ab["draft_rows"] == 3
    assert ab["target_rows"] == 6
    assert ab["draft_bytes"] == 3 * 100 * 4
    assert ab["target_bytes"] == 6 * 300 * 2
    assert ab["total"] == 1200 + 3600


def _summary(path, sha, traffic, top_k=None):
    lines = ["# a summary", "", "- source_sha256: `%s`" % sha]
    if top_k is not None:
        lines.append("- top_k: %d" % top_k)
    lines.append("- traffic_bytes_per_launch: %d" % traffic)
    path.write_text("\n".join(lines) + "\n")


def test_traffic_only_from_a_summary_of_the_current_source(tmp_path, monkeypatch):
    (tmp_path / "profiles").mkdir()
    monkeypatch.setattr(bench, "ROOT", str(tmp_path))
    monkeypatch.setattr(bench, "rowpass_source_hash", lambda: "0123456789abcdef")
    assert bench.profiled_traffic("wl") is None  # no summary
    _summary(tmp_path / "profiles" / "rowpass_wl.md", "0123456789abcdef", 123456)
    assert bench.profiled_traffic("wl") == 123456.0
    _summary(tmp_path / "profiles" / "rowpass_wl.md", "fedcba9876543210", 123456)
    assert bench.profiled_traffic("wl") is None  # taken on another source
    # filtered runs read their own summary, only at the top-k it was taken at
    assert bench.profiled_traffic("wl", 20) is None
    _summary(tmp_path / "profiles" / "rowpass_filtered_wl.md", "0123456789abcdef", 777, 20)
    assert bench.profiled_traffic("wl", 20) == 777.0
    assert bench.profiled_traffic("wl", 10) is None


def test_source_hash_covers_the_row_pass_sources():
    for rel in bench.ROWPASS_SOURCES:
        assert os.path.isfile(os.path.join(ROOT, rel)), rel
    h = bench.rowpass_source_hash()
    assert len(h) == 16 and int(h, 16) >= 0


def test_reference_arm_prints_one_contract_line():
    env = dict(os.environ, CUDA_VISIBLE_DEVICES="")
    r = subprocess.run([sys.executable, "bench.py", "--impl", "reference", "--workload",
                        "b1_g4_v32k", "--steps", "2", "--warmup", "3"], cwd=ROOT, env=env,
                       capture_output=True, text=True, timeout=600)
    assert r.returncode == 0, r.stderr[-2000:]
    lines = [l for l in r.stdout.splitlines() if l.startswith("{")]
    assert len(lines) == 1
    d = json.loads(lines[0])
    assert d["impl"] == "reference" and d["metric"] == bench.METRIC and d["unit"] == bench.UNIT
    assert d["value"] > 0 and d["steps"] == 2 and d["warmup"] >= 3 and d["n_gpus"] == 1
    assert d["higher_is_better"] is True and d["config"]["workload"] == "b1_g4_v32k"
    # the workload keys of the GPU arm's config (its measured keys aside)
    for key in ("batch_per_gpu", "gamma", "V_d", "V_t", "logits_cols", "target_tokens_per_gpu",
                "window", "temperature", "filters", "parallelism"):
        assert key in d["config"], key
    assert d["config"]["batch_per_gpu"] == 1 and d["config"]["gamma"] == 4
    assert d["config"]["filters"] is None
    cb = d["cpu_baseline"]
    assert cb["kind"] == "oracle" and cb["cores"] >= 1 and cb["value"] == d["value"]
    assert d["e2e"] == {"value": d["value"], "unit": d["unit"], "h2d_bytes_per_step": 0,
                        "d2h_bytes_per_step": 0}


@pytest.mark.parametrize("window", [-1, 0, 1, 2, 8])
def test_band_cells_match_a_count_of_the_band(window):
    rng = np.random.default_rng(window + 5)
    k = rng.integers(1, 30, size=40)
    m = rng.integers(1, 30, size=40)
    wl = SimpleNamespace(draft_off=np.concatenate([[0], np.cumsum(k)]),
                         target_off=np.concatenate([[0], np.cumsum(m)]))
    want = 0
    for kb, mb in zip(k, m):
        W = max(window, abs(int(kb) - int(mb)))
        want += sum(1 for i in range(1, kb + 1) for j in range(1, mb + 1)
                    if window < 0 or abs(i - j) <= W)
    assert bench.band_cells(wl, window) == want
    # the band always holds the diagonal corner to corner, at most every cell
    assert int((np.minimum(k, m)).sum()) <= bench.band_cells(wl, window) <= int((k * m).sum())


def test_oracle_legs_run_the_step_parameters_of_the_run(monkeypatch):
    """The CPU legs time the oracle on the run's temperature and filters."""
    import oracle
    from paper_2510_15545_gb300 import workload as W
    seen = []
    real = oracle.step

    def spy(sw, **kw):
        seen.append(kw)
        return real(sw, **kw)
    monkeypatch.setattr(oracle, "step", spy)
    wl = W.make_workload("b1_g4_v32k", seed=0)
    args = bench.parse_args(["--temp", "0.6", "--top-k", "20", "--top-p", "0.95"])
    rate, sample, n, el = bench.oracle_sample_rate(wl, 0.05, bench.step_kwargs(args))
    assert rate > 0 and n >= 1
    assert seen and all(k["temp_draft"] == 0.6 and k["temp_target"] == 0.6 and
                        k["top_k_draft"] == 20 and k["top_p_target"] == 0.95 for k in seen)
    plain = bench.step_kwargs(bench.parse_args([]))
    assert plain == {"top_k_draft": 0, "top_k_target": 0, "top_p_draft": 1.0,
                     "top_p_target": 1.0}
    # a worker job carries the same parameters
    pos, sec, done = bench._oracle_job(([(0, wl.subset([0]))], 0.0, bench.step_kwargs(args)))
    assert done == 1 and pos == 4 and seen[-1]["top_k_target"] == 20


def test_cpu_leg_counts_boundary_cases_and_mismatches(monkeypatch):
    """The CPU-baseline leg compares its oracle sample with the device step's
    outputs for the same requests: the oracle against itself gives no
    mismatch; a planted wrong next token is counted as one."""
    import oracle
    import torch
    from paper_2510_15545_gb300 import workload as W
    monkeypatch.setattr(bench, "oracle_all_cores_rate", lambda wl, b, step_kw=None: (1.0, "-", 1))
    wl = W.make_workload("b1_g4_v32k", B=3, seed=2)
    o = oracle.step(wl)
    keys = ("status", "accepted", "next_token", "path_len", "cost", "map", "q_hat", "p_hat", "lse")
    full = {k: torch.as_tensor(np.asarray(o[k])) for k in keys}
    full["path"] = torch.as_tensor(np.asarray(o["path"]).ravel())
    args = bench.parse_args(["--cpu-seconds", "0.05"])
    cpu, cpu_all, bnd = bench.cpu_baseline_leg(wl, full, args, bench.step_kwargs(args))
    assert cpu["cores"] == 1 and cpu["kind"] == "oracle"
    assert bnd["requests_compared"] == 3 and bnd["mismatches"] == 0
    full["next_token"][1] = (int(o["next_token"][1]) + 7) % wl.target_logits.shape[1]
    cpu, cpu_all, bnd = bench.cpu_baseline_leg(wl, full, args, bench.step_kwargs(args))
    assert bnd["mismatches"] == 1 and bnd["first_mismatches"]


def test_launch_count_traffic_and_filters_key_follow_the_run_filters():
    """gpu_launches counts the kernels each filter family launches (nucleus:
    merge and exact kernels; penalty: its per-request sets), and only runs
    whose row-pass variant has a committed summary may carry its traffic."""
    p = bench.parse_args
    assert bench.step_launches(p([])) == 3
    assert bench.step_launches(p(["--top-k", "20", "--top-p", "0.95"])) == 5
    assert bench.step_launches(p(["--top-p", "0.9"])) == 6
    assert bench.step_launches(p(["--top-k", "20", "--rep-penalty", "1.1"])) == 6
    assert bench.run_traffic("no_such_workload", p(["--top-p", "0.9"])) is None
    assert bench.run_traffic("no_such_workload",
                             p(["--top-k", "20", "--rep-penalty", "1.1"])) is None
    assert bench.filters_config(p([])) is None
    assert bench.filters_config(p(["--top-p", "0.9"])) == {"top_k": 0, "top_p": 0.9}
    f = bench.filters_config(p(["--top-k", "20", "--rep-penalty", "1.1"]))
    assert f["rep_penalty"] == 1.1 and f["top_k"] == 20
    kw = bench.step_kwargs(p(["--top-k", "20", "--rep-penalty", "1.1"]))
    assert kw["rep_penalty_draft"] == kw["rep_penalty_target"] == 1.1
