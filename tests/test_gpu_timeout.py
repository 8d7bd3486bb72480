"""Failure detection without a GPU fault: every pipeline wait of the row pass is
bounded in time. A test hook, read by the library once per process from the
environment (TT_TEST_STALL_STAGE, TT_TEST_WAIT_MS), makes one CTA of the
process's first row-pass launch hold one stage and lowers that launch's limit
to 50 ms, so its waits run out: the call must end on its own, report
TT_REQ_TIMEOUT for every request (accepted 0, next token -1), and leave the
context usable -- the next call in the same process, which the hook no longer
touches, matches the oracle. Each case runs in a child process of its own, so
the hook reaches no other test."""
import os
import subprocess
import sys

import pytest
import torch

pytestmark = pytest.mark.gpu

HERE = os.path.dirname(os.path.abspath(__file__))
ROOT = os.path.dirname(HERE)

CHILD = r"""
import sys, time
sys.path.insert(0, %(root)r)
sys.path.insert(0, %(here)r)
import numpy as np
import paper_2510_15545_gb300 as tt
from paper_2510_15545_gb300 import binding
from paper_2510_15545_gb300 import workload as W
from _parity import compare, gpu_step, oracle_step
tt.load(build_if_missing=True)
f = %(filters)r
wl = W.make_workload(%(name)r, B=8, seed=%(seed)d)
t0 = time.perf_counter()
g = gpu_step(wl, **f)
elapsed = time.perf_counter() - t0
assert np.all((g["status"] & 32) != 0), g["status"]
assert np.all(g["accepted"] == 0) and np.all(g["next_token"] == -1)
assert elapsed < 20.0, elapsed
assert binding.load().tt_last_cuda_error() == 0
g2 = gpu_step(wl, **f)
compare(wl, g2, oracle_step(wl, **f))
print("child ok")
"""


def _run_child(name, seed, stage, filters):
    if not torch.cuda.is_available():
        pytest.skip("needs a GPU")
    env = dict(os.environ, TT_TEST_STALL_STAGE=str(stage), TT_TEST_WAIT_MS="50")
    code = CHILD % dict(root=ROOT, here=HERE, filters=filters, name=name, seed=seed)
    p = subprocess.run([sys.executable, "-c", code], env=env, capture_output=True, text=True,
                       timeout=600)
    assert p.returncode == 0 and "child ok" in p.stdout, (p.stdout[-2000:], p.stderr[-4000:])


@pytest.mark.parametrize("name", ["b64_g8_v152k", "b1024_g8_v201k_bf16"])
def test_bounded_waits_run_out_and_the_context_stays_usable(name):
    _run_child(name, 5, 2, {})


def test_filtered_step_reports_the_timeout():
    f = dict(temp_draft=0.6, temp_target=0.6, top_k_draft=20, top_p_draft=0.95,
             top_k_target=20, top_p_target=0.95)
    _run_child("b64_g8_v152k", 6, 3, f)
