"""Failure detection without a GPU fault: every pipeline wait of the row pass is
bounded in time. A test hook (TT_TEST_STALL_STAGE, TT_TEST_WAIT_MS, read by the
library at each row-pass launch) makes one CTA hold one stage and lowers the
limit to 50 ms, so the waits run out: the call must end on its own, report
TT_REQ_TIMEOUT for every request (accepted 0, next token -1), and leave the
context usable -- the next call, without the hook, matches the oracle."""
import time

import numpy as np
import pytest
import torch

import paper_2510_15545_gb300 as tt
from paper_2510_15545_gb300 import binding
from paper_2510_15545_gb300 import workload as W
from _parity import compare, gpu_step, oracle_step

pytestmark = pytest.mark.gpu

TT_REQ_TIMEOUT = 32


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.skip("needs a GPU")
    tt.load(build_if_missing=True)


@pytest.mark.parametrize("name", ["b64_g8_v152k", "b1024_g8_v201k_bf16"])
def test_bounded_waits_run_out_and_the_context_stays_usable(monkeypatch, name):
    wl = W.make_workload(name, B=8, seed=5)
    monkeypatch.setenv("TT_TEST_STALL_STAGE", "2")
    monkeypatch.setenv("TT_TEST_WAIT_MS", "50")
    t0 = time.perf_counter()
    g = gpu_step(wl)
    elapsed = time.perf_counter() - t0
    assert np.all((g["status"] & TT_REQ_TIMEOUT) != 0), g["status"]
    assert np.all(g["accepted"] == 0) and np.all(g["next_token"] == -1)
    assert elapsed < 20.0
    assert binding.load().tt_last_cuda_error() == 0
    monkeypatch.delenv("TT_TEST_STALL_STAGE")
    monkeypatch.delenv("TT_TEST_WAIT_MS")
    g2 = gpu_step(wl)
    compare(wl, g2, oracle_step(wl))


def test_filtered_step_reports_the_timeout(monkeypatch):
    wl = W.make_workload("b64_g8_v152k", B=8, seed=6)
    f = dict(temp_draft=0.6, temp_target=0.6, top_k_draft=20, top_p_draft=0.95,
             top_k_target=20, top_p_target=0.95)
    monkeypatch.setenv("TT_TEST_STALL_STAGE", "3")
    monkeypatch.setenv("TT_TEST_WAIT_MS", "50")
    g = gpu_step(wl, **f)
    assert np.all((g["status"] & TT_REQ_TIMEOUT) != 0), g["status"]
    assert np.all(g["next_token"] == -1)
    monkeypatch.delenv("TT_TEST_STALL_STAGE")
    monkeypatch.delenv("TT_TEST_WAIT_MS")
    g2 = gpu_step(wl, **f)
    compare(wl, g2, oracle_step(wl, **f))
