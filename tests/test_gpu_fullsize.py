"""Parity at full workload size, in the launch configuration the benchmark
times (one tt_step over the whole batch): the oracle recomputes a sample of
requests one by one (with their global Philox request index), and properties
that hold at any size are checked on every request."""
import numpy as np
import pytest
import torch

import oracle
import paper_2510_15545_gb300 as tt
from paper_2510_15545_gb300 import workload as W

from _parity import compare, oracle_step, sub_workload, to_np

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.skip("needs a GPU")
    tt.load(build_if_missing=True)


@pytest.mark.parametrize("name,n_sample", [("b64_g8_v152k", 10), ("b256_g16_v152k_bf16", 12),
                                           ("b1024_g8_v201k_bf16", 6), ("dtw_4096x64", 12)])
def test_full_size_step_sampled(name, n_sample):
    """One full-size tt_step as the benchmark launches it (the decision kernel
    at 256 threads per request, or 128 for the 1024-request and the
    4096-request DTW batches): every request's invariants, a sample against
    the oracle."""
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
    total = dict(accept_boundary=0, token_boundary=0, filter_boundary=0)
    for b in idx:
        sw = sub_workload(wl, [b])
        o = oracle_step(sw, request_base=int(b))
        g = {k: v for k, v in out.items()}
        g["_target_off"], g["_draft_off"] = wl.target_off, wl.draft_off
        c = compare(sw, g, o, req_index=[b])
        for key in total:
            total[key] += c[key]
    print(name, "sampled", len(idx), total)


FILTERS = dict(temp_draft=0.6, temp_target=0.6, top_k_draft=20, top_p_draft=0.95,
               top_k_target=20, top_p_target=0.95)


@pytest.mark.parametrize("name,n_sample", [("b64_g8_v152k", 10), ("b1024_g8_v201k_bf16", 6)])
def test_full_size_filtered_step_sampled(name, n_sample):
    """The paper's Qwen3 sampling setting on both families, full batch, one
    tt_step as the benchmark times it; a sample of requests against the oracle."""
    wl = W.make_workload(name, seed=0, device="cuda")
    inp = tt.device_inputs(wl, "cuda")
    prm = inp["params"]
    for k, v in FILTERS.items():
        setattr(prm, k, v)
    out = to_np(tt.tt_step(inp["batch"], inp["vd"], inp["vt"], inp["draft_logits"],
                           inp["target_logits"], prm))
    m = np.diff(wl.target_off)
    assert np.all(out["status"] == 0)
    assert np.all((out["accepted"] >= 0) & (out["accepted"] <= m))
    assert np.all((out["next_token"] >= 0) & (out["next_token"] < wl.target_logits.shape[1]))
    assert np.all((out["p_hat"] >= 0) & (out["p_hat"] <= 1))
    assert np.all((out["q_hat"] >= 0) & (out["q_hat"] <= 1))
    rng = np.random.default_rng(2)
    B = wl.B
    idx = np.unique(np.concatenate([[0, B - 1], rng.choice(B, size=n_sample, replace=False)]))
    for b in idx:
        sw = sub_workload(wl, [b])
        o = oracle_step(sw, request_base=int(b), **FILTERS)
        g = dict(out)
        g["_target_off"], g["_draft_off"] = wl.target_off, wl.draft_off
        compare(sw, g, o, req_index=[b])


def test_full_size_sharded_verify_sampled():
    """tt_verify_sharded over the full 1024-request bf16 batch in four shards,
    q_hat from the step: a sample against the oracle, every request against
    the unsplit verification."""
    wl = W.make_workload("b1024_g8_v201k_bf16", seed=0, device="cuda")
    inp = tt.device_inputs(wl, "cuda")
    prm = inp["params"]
    step = tt.tt_step(inp["batch"], inp["vd"], inp["vt"], inp["draft_logits"],
                      inp["target_logits"], prm)
    tl = inp["target_logits"]
    V = tl.shape[1]
    cuts = [0, 50000, 100001, 150007, V]
    shards = []
    for a, b in zip(cuts, cuts[1:]):
        buf = torch.empty((tl.shape[0], (b - a + 7) // 8 * 8), dtype=tl.dtype, device="cuda")
        buf[:, :b - a] = tl[:, a:b]
        shards.append(buf[:, :b - a])
    g = to_np(tt.tt_verify_sharded(inp["batch"], step["q_hat"], shards, prm))
    u = to_np(tt.tt_verify(inp["batch"], step["q_hat"], tl, prm))
    assert np.all(g["status"] == 0)
    assert np.array_equal(g["accepted"], u["accepted"])
    assert np.max(np.abs(g["p_hat"] - u["p_hat"])) <= 1e-5
    # tokens may differ only where the residual's running mass meets the draw
    # within rounding (a handful of requests at most)
    assert int((g["next_token"] != u["next_token"]).sum()) <= 8
    q = step["q_hat"].cpu().numpy()
    rng = np.random.default_rng(3)
    for b in np.unique(np.concatenate([[0, wl.B - 1], rng.choice(wl.B, size=6, replace=False)])):
        sw = sub_workload(wl, [b])
        t0, t1 = int(wl.target_off[b]), int(wl.target_off[b + 1])
        o = oracle.verify(sw.target_off, sw.target_cols, q[t0:t1].astype(np.float64),
                          sw.target_logits, temp_target=prm.temp_target, seed=prm.seed,
                          request_base=int(b))
        gg = {k: v for k, v in g.items()}
        gg["q_hat"] = q
        gg["_target_off"], gg["_draft_off"] = wl.target_off, wl.draft_off
        oo = dict(o)
        oo["q_hat"] = q[t0:t1]
        compare(sw, gg, oo, req_index=[b], check_align=False)


def test_full_size_alignment_alone_and_in_step():
    """All 4096 pairs of the DTW workload (64 draft tokens, 48..96 target
    tokens each) against the oracle, in both launch shapes of the alignment
    kernel: tt_align alone (one warp per pair, more CTAs than SMs) and inside
    tt_step (one CTA per SM, its warps looping over about 27 pairs each)."""
    wl = W.make_workload("dtw_4096x64", seed=0, device="cuda")
    inp = tt.device_inputs(wl, "cuda")
    prm = inp["params"]
    o = oracle.align(wl.draft_off, wl.draft_ids, wl.target_off, wl.target_ids, wl.vd.blob,
                     wl.vd.off, wl.vt.blob, wl.vt.off, prm.window)
    alone = to_np(tt.tt_align(inp["batch"], inp["vd"], inp["vt"], prm))
    step = to_np(tt.tt_step(inp["batch"], inp["vd"], inp["vt"], inp["draft_logits"],
                            inp["target_logits"], prm))
    torch.cuda.synchronize()
    assert np.all(o["status"] == 0)
    for g in (alone, step):
        assert np.array_equal(g["status"], o["status"])
        assert np.array_equal(g["path_len"], o["path_len"])
        assert np.array_equal(g["cost"], o["cost"])
        assert np.array_equal(g["map"], o["map"])
        for b in range(wl.B):
            p0 = int(wl.draft_off[b] + wl.target_off[b])
            L = int(o["path_len"][b])
            assert np.array_equal(g["path"][2 * p0:2 * (p0 + L)], o["path"][p0:p0 + L].ravel())
