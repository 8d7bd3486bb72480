"""GPU parity of top-p without top-k (the nucleus rows of the paper's
generation hyperparameter table, App. F: the Llama-3.1-70B target at T = 0.6,
top-p 0.9 and the DeepSeek-R1-Distill-Llama-70B target at T = 0.6, top-p 0.95)
against the oracle, through the C ABI: tt_step with nucleus target rows, draft
rows or both, beside top-k families; nuclei from a handful of columns to well
over the 32 a top-k list holds; rows of many tied logits and rows where one
logit takes nearly all the mass; tt_transfer and tt_verify alone; full-size
batches in the benchmark's launch configuration."""
import dataclasses

import numpy as np
import pytest
import torch

import oracle
import paper_2510_15545_gb300 as tt
from paper_2510_15545_gb300 import workload as W
from _parity import compare, gpu_step, oracle_step, sub_workload, to_np

pytestmark = pytest.mark.gpu
_CACHE = {}

LLAMA = dict(temp_draft=0.6, temp_target=0.6, top_p_draft=0.9, top_p_target=0.9)
DEEPSEEK = dict(temp_draft=0.6, temp_target=0.6, top_p_draft=0.95, top_p_target=0.95)


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.skip("needs a GPU")
    tt.load(build_if_missing=True)


def _wl(name, B, seed=0):
    return W.make_workload(name, B=B, seed=seed, vocab_cache=_CACHE)


def _nucleus_sizes(wl, T, p):
    z = wl.target_logits.float().numpy().astype(np.float64) / T
    z -= z.max(1, keepdims=True)
    e = np.exp(z)
    e /= e.sum(1, keepdims=True)
    srt = -np.sort(-e, axis=1)
    return ((np.cumsum(srt, axis=1) - srt) < p).sum(1)


@pytest.mark.parametrize("f", [LLAMA, DEEPSEEK], ids=["llama_p090", "deepseek_p095"])
@pytest.mark.parametrize("name,B", [("b64_g8_v152k", 12), ("b1024_g8_v201k_bf16", 8),
                                    ("b256_g16_v152k_bf16", 4), ("dtw_4096x64", 6),
                                    ("b1_g4_v32k", 1)])
def test_nucleus_step_matches_oracle(f, name, B):
    wl = _wl(name, B, seed=3)
    g = gpu_step(wl, **f)
    o = oracle_step(wl, **f)
    r = compare(wl, g, o)
    assert r["filter_boundary"] <= B // 4, r


def test_nuclei_beyond_a_top_k_list_are_covered():
    """The test rows above include nuclei much larger than 32 columns."""
    wl = _wl("b1024_g8_v201k_bf16", 8, seed=3)
    n = _nucleus_sizes(wl, 0.6, 0.95)
    assert n.max() > 100 and (n > 32).mean() > 0.3, n


@pytest.mark.parametrize("f", [
    dict(temp_target=0.6, top_p_target=0.9),                                   # target only
    dict(temp_draft=0.6, top_p_draft=0.95),                                    # draft only
    dict(temp_draft=0.7, top_k_draft=20, top_p_draft=0.8, temp_target=0.6,
         top_p_target=0.95),                                                   # Qwen2.5 draft, DeepSeek target
    dict(temp_draft=0.6, top_p_draft=0.9, temp_target=0.6, top_k_target=20,
         top_p_target=0.95),                                                   # nucleus draft, Qwen3 target
    dict(temp_draft=1.3, top_p_draft=0.5, temp_target=0.4, top_p_target=0.99),
])
def test_nucleus_beside_other_families(f):
    for name, B in (("b64_g8_v152k", 10), ("b1024_g8_v201k_bf16", 6)):
        wl = _wl(name, B, seed=7)
        compare(wl, gpu_step(wl, **f), oracle_step(wl, **f))


def test_ties_and_a_dominant_logit():
    """Rows of coarse integer logits (long runs of ties at the cut) and rows
    where one logit holds nearly all the mass (a nucleus of one column)."""
    wl = _wl("b64_g8_v152k", 8, seed=11)
    rng = np.random.default_rng(5)
    tl = torch.as_tensor(rng.integers(-3, 4, size=wl.target_logits.shape).astype(np.float32))
    dl = torch.as_tensor(rng.integers(-3, 4, size=wl.draft_logits.shape).astype(np.float32))
    tl[::3, 17] = 60.0  # every third target row: one dominant column
    wl2 = dataclasses.replace(wl, target_logits=tl, draft_logits=dl)
    for f in (LLAMA, DEEPSEEK, dict(temp_draft=1.0, top_p_draft=0.3, temp_target=1.0,
                                     top_p_target=0.3)):
        compare(wl2, gpu_step(wl2, **f), oracle_step(wl2, **f))


def _padded(t: torch.Tensor) -> torch.Tensor:
    """``t`` on the GPU as a view into rows padded to a 16-byte multiple plus
    one more 16-byte vector, the padding NaN: a read past a row's end shows."""
    R, V = t.shape
    per16 = 16 // t.element_size()
    buf = torch.full((R, (V + per16 - 1) // per16 * per16 + per16), float("nan"),
                     dtype=t.dtype, device="cuda")
    buf[:, :V] = t.to("cuda")
    return buf[:, :V]


@pytest.mark.parametrize("V,dtype", [(37, torch.float32), (4100, torch.float32),
                                     (2053, torch.bfloat16), (6001, torch.bfloat16)])
def test_narrow_and_ragged_rows(V, dtype):
    """Rows narrower than a chunk or with a ragged tail, their padding NaN."""
    wl = W.homogeneous_workload(6, 4, V, seed=V, dtype=dtype)
    inp = tt.device_inputs(wl, "cuda")
    prm = inp["params"]
    for k, v in DEEPSEEK.items():
        setattr(prm, k, v)
    g = to_np(tt.tt_step(inp["batch"], inp["vd"], inp["vt"], _padded(wl.draft_logits),
                         _padded(wl.target_logits), prm))
    compare(wl, g, oracle_step(wl, **DEEPSEEK))


def test_transfer_and_verify_alone_with_nucleus_rows():
    wl = _wl("b64_g8_v152k", 16, seed=5)
    inp = tt.device_inputs(wl, "cuda")
    prm = inp["params"]
    prm.temp_draft = prm.temp_target = 0.6
    prm.top_p_draft, prm.top_p_target = 0.95, 0.9
    al = oracle.align(wl.draft_off, wl.draft_ids, wl.target_off, wl.target_ids, wl.vd.blob,
                      wl.vd.off, wl.vt.blob, wl.vt.off, wl.spec.window)
    mp = torch.as_tensor(al["map"], dtype=torch.int32, device="cuda")
    tr = to_np(tt.tt_transfer(inp["batch"], mp, prm, draft_logits=inp["draft_logits"]))
    otr = oracle.transfer(wl.draft_off, wl.draft_cols, wl.target_off, al["map"], wl.draft_logits,
                          0.6, top_k=0, top_p=0.95)
    assert np.array_equal(tr["status"][:wl.B], otr["status"])
    amb = otr["drow_bnd"][wl.draft_off[:-1].repeat(np.diff(wl.target_off)) + al["map"]] & 4
    ok = amb == 0
    d = np.abs(tr["q_hat"][:wl.n_target] - otr["q_hat"])
    assert np.all((d[ok] <= 1e-5) & (d[ok] <= 1e-4 * otr["q_hat"][ok] + 1e-30))
    q = torch.as_tensor(otr["q_hat"], dtype=torch.float32, device="cuda")
    ve = to_np(tt.tt_verify(inp["batch"], q, inp["target_logits"], prm))
    ove = oracle.verify(wl.target_off, wl.target_cols, otr["q_hat"], wl.target_logits,
                        temp_target=0.6, seed=prm.seed, top_k_target=0, top_p_target=0.9)
    g = dict(ve)
    g["q_hat"] = otr["q_hat"]
    o = dict(ove)
    o["q_hat"] = otr["q_hat"]
    compare(wl, g, o, check_align=False)


@pytest.mark.parametrize("name,n_sample", [("b64_g8_v152k", 8), ("b1024_g8_v201k_bf16", 5)])
def test_full_size_nucleus_step_sampled(name, n_sample):
    """The DeepSeek setting on both families, full batch, one tt_step as the
    benchmark times it: every request's invariants, a sample against the oracle."""
    wl = W.make_workload(name, seed=0, device="cuda")
    inp = tt.device_inputs(wl, "cuda")
    prm = inp["params"]
    for k, v in DEEPSEEK.items():
        setattr(prm, k, v)
    out = to_np(tt.tt_step(inp["batch"], inp["vd"], inp["vt"], inp["draft_logits"],
                           inp["target_logits"], prm))
    m = np.diff(wl.target_off)
    assert np.all(out["status"] == 0)
    assert np.all((out["accepted"] >= 0) & (out["accepted"] <= m))
    assert np.all((out["next_token"] >= 0) & (out["next_token"] < wl.target_logits.shape[1]))
    assert np.all((out["p_hat"] >= 0) & (out["p_hat"] <= 1))
    rng = np.random.default_rng(4)
    B = wl.B
    for b in np.unique(np.concatenate([[0, B - 1], rng.choice(B, size=n_sample, replace=False)])):
        sw = sub_workload(wl, [b])
        o = oracle_step(sw, request_base=int(b), **DEEPSEEK)
        g = dict(out)
        g["_target_off"], g["_draft_off"] = wl.target_off, wl.draft_off
        compare(sw, g, o, req_index=[b])


def crowded_rows(wl, seed=21):
    """Target logits whose rows hold a small nucleus near the maximum (a column
    at 0 and a few within 3 log2 units at T = 0.6) and 5000 columns between 12.5
    and 13.5 log2 units below it, the rest far below: at top-p 0.5 the cut lies
    in the nucleus, while more than 4096 columns lie within 14 units."""
    rng = np.random.default_rng(seed)
    R, V = wl.target_logits.shape
    scale = 1.4426950408889634 / 0.6
    z = np.full((R, V), -40.0, np.float32)
    for r in range(R):
        cols = rng.permutation(V)
        z[r, cols[0]] = 0.0
        z[r, cols[1:5]] = -rng.uniform(0.5, 3.0, 4) / scale
        z[r, cols[5:5005]] = -rng.uniform(12.5, 13.5, 5000) / scale
    return dataclasses.replace(wl, target_logits=torch.as_tensor(z))


def test_rows_that_overflow_the_first_candidate_bar():
    """The nucleus kernel's second candidate pass (a lower whole bar estimated
    from the held candidates) settles these rows; compared with the oracle."""
    wl = crowded_rows(_wl("b64_g8_v152k", 6, seed=13))
    f = dict(temp_target=0.6, top_p_target=0.5)
    compare(wl, gpu_step(wl, **f), oracle_step(wl, **f))
