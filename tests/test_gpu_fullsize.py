"""Parity at full workload size, in the launch configuration the benchmark
times (one tt_step over the whole batch): the oracle recomputes a sample of
requests one by one (with their global Philox request index), and properties
that hold at any size are checked on every request."""
import numpy as np
import pytest
import torch

import paper_2510_15545_gb300 as tt
from paper_2510_15545_gb300 import workload as W

from _parity import compare, oracle_step, sub_workload, to_np

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.skip("needs a GPU")
    tt.load(build_if_missing=True)


@pytest.mark.parametrize("name,n_sample", [("b64_g8_v152k", 10), ("b1024_g8_v201k_bf16", 6)])
def test_full_size_step_sampled(name, n_sample):
    wl = W.make_workload(name, seed=0, device="cuda")
    inp = tt.device_inputs(wl, "cuda")
    out = to_np(tt.tt_step(inp["batch"], inp["vd"], inp["vt"], inp["draft_logits"],
                           inp["target_logits"], inp["params"]))
    torch.cuda.synchronize()
    B = wl.B
    # any size: every request succeeded, accepted within 0..m, tokens in range,
    # probabilities in [0, 1], the path ends at (k-1, m-1)
    m = np.diff(wl.target_off)
    assert np.all(out["status"] == 0)
    assert np.all((out["accepted"] >= 0) & (out["accepted"] <= m))
    assert np.all((out["next_token"] >= 0) & (out["next_token"] < wl.target_logits.shape[1]))
    assert np.all((out["p_hat"] >= 0) & (out["p_hat"] <= 1))
    assert np.all((out["q_hat"] >= 0) & (out["q_hat"] <= 1))
    for b in range(B):
        p0 = int(wl.draft_off[b] + wl.target_off[b])
        L = int(out["path_len"][b])
        last = out["path"][2 * (p0 + L - 1):2 * (p0 + L)]
        assert list(last) == [int(wl.draft_off[b + 1] - wl.draft_off[b]) - 1, int(m[b]) - 1]
    # a sample of requests, one by one, against the oracle
    rng = np.random.default_rng(1)
    idx = np.unique(np.concatenate([[0, B - 1], rng.choice(B, size=n_sample, replace=False)]))
    total = dict(accept_boundary=0, token_boundary=0)
    for b in idx:
        sw = sub_workload(wl, [b])
        o = oracle_step(sw, request_base=int(b))
        g = {k: v for k, v in out.items()}
        g["_target_off"], g["_draft_off"] = wl.target_off, wl.draft_off
        c = compare(sw, g, o, req_index=[b])
        for key in total:
            total[key] += c[key]
    print(name, "sampled", len(idx), total)
