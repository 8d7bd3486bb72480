"""GPU parity of the repetition penalty (the generation hyperparameter table,
App. F: the Qwen2.5-0.5B row, T = 0.7, top-p 0.8, top-k 20, penalty 1.1)
against the oracle, through the C ABI: both families or one, other penalties
(one below 1 too), histories with repeats, empty or absent histories, rows
whose penalized columns lead the row, the statuses of bad histories, the
argument rules, tt_transfer and tt_verify alone, and full-size batches in the
benchmark's launch configuration."""
import numpy as np
import pytest
import torch

import oracle
import paper_2510_15545_gb300 as tt
from paper_2510_15545_gb300 import workload as W
from _parity import compare, gpu_step, oracle_step, sub_workload, to_np

pytestmark = pytest.mark.gpu
_CACHE = {}

QWEN25 = dict(temp_draft=0.7, temp_target=0.7, top_k_draft=20, top_p_draft=0.8,
              top_k_target=20, top_p_target=0.8, rep_penalty_draft=1.1, rep_penalty_target=1.1)


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.skip("needs a GPU")
    tt.load(build_if_missing=True)


def _wl(name, B, seed=0, lo=20, hi=400):
    return W.with_histories(W.make_workload(name, B=B, seed=seed, vocab_cache=_CACHE), lo, hi,
                            seed=seed)


@pytest.mark.parametrize("name,B", [("b64_g8_v152k", 12), ("b1024_g8_v201k_bf16", 8),
                                    ("b256_g16_v152k_bf16", 4), ("dtw_4096x64", 6),
                                    ("b1_g4_v32k", 1)])
def test_qwen25_setting_matches_oracle(name, B):
    wl = _wl(name, B, seed=2)
    compare(wl, gpu_step(wl, **QWEN25), oracle_step(wl, **QWEN25))


@pytest.mark.parametrize("f", [
    dict(temp_draft=0.7, top_k_draft=20, top_p_draft=0.8, rep_penalty_draft=1.1),   # draft only
    dict(temp_target=0.7, top_k_target=20, top_p_target=0.8, rep_penalty_target=1.1),
    dict(top_k_draft=32, top_k_target=32, rep_penalty_draft=1.5, rep_penalty_target=2.0),
    dict(top_k_draft=5, top_k_target=8, top_p_target=0.9, rep_penalty_draft=0.8,
         rep_penalty_target=0.7),                                                    # below 1
    dict(top_k_draft=20, top_p_draft=0.8, top_k_target=20, top_p_target=0.8,
         rep_penalty_target=1.1),                                                    # filters, one penalty
])
def test_other_penalties_and_families(f):
    for name, B in (("b64_g8_v152k", 10), ("b1024_g8_v201k_bf16", 6)):
        wl = _wl(name, B, seed=5)
        compare(wl, gpu_step(wl, **f), oracle_step(wl, **f))


def test_histories_absent_empty_long_and_repeated():
    wl = W.make_workload("b64_g8_v152k", B=8, seed=9, vocab_cache=_CACHE)
    # no histories at all: only the sequence tokens before each row are penalized
    compare(wl, gpu_step(wl, **QWEN25), oracle_step(wl, **QWEN25))
    # empty histories, one history repeating one column, one at the cap
    V_t, V_d = wl.target_logits.shape[1], wl.draft_logits.shape[1]
    rng = np.random.default_rng(3)
    lens = [0, 50, 0, 3072,
            7, 0, 300, 1]
    rep = [None, 11, None, None, None, None, None, None]
    hot, hct, hod, hcd = [0], [], [0], []
    for n, r in zip(lens, rep):
        t = np.full(n, r, np.int32) if r is not None else rng.integers(0, V_t, n).astype(np.int32)
        d = rng.integers(0, V_d, n).astype(np.int32)
        hct.append(t)
        hcd.append(d)
        hot.append(hot[-1] + n)
        hod.append(hod[-1] + n)
    wl2 = W.Workload(**{**wl.__dict__, "hist_off_t": np.array(hot, np.int32),
                        "hist_cols_t": np.concatenate(hct), "hist_off_d": np.array(hod, np.int32),
                        "hist_cols_d": np.concatenate(hcd)})
    compare(wl2, gpu_step(wl2, **QWEN25), oracle_step(wl2, **QWEN25))


def test_penalized_columns_that_lead_their_rows():
    """Histories made of each row's largest logits: the penalized columns are
    the rows' top candidates, so the merge of the lists with the penalized
    columns decides the top-k."""
    wl = W.make_workload("b1024_g8_v201k_bf16", B=6, seed=4, vocab_cache=_CACHE)
    hot, hct, hod, hcd = [0], [], [0], []
    for b in range(wl.B):
        r0, r1 = int(wl.target_off[b]) + b, int(wl.target_off[b + 1]) + b + 1
        top_t = torch.topk(wl.target_logits[r0:r1].float(), 12, dim=1).indices.flatten()
        d0, d1 = int(wl.draft_off[b]), int(wl.draft_off[b + 1])
        top_d = torch.topk(wl.draft_logits[d0:d1].float(), 12, dim=1).indices.flatten()
        hct.append(top_t.numpy().astype(np.int32))
        hcd.append(top_d.numpy().astype(np.int32))
        hot.append(hot[-1] + len(hct[-1]))
        hod.append(hod[-1] + len(hcd[-1]))
    wl2 = W.Workload(**{**wl.__dict__, "hist_off_t": np.array(hot, np.int32),
                        "hist_cols_t": np.concatenate(hct), "hist_off_d": np.array(hod, np.int32),
                        "hist_cols_d": np.concatenate(hcd)})
    for f in (QWEN25, dict(QWEN25, top_k_draft=3, top_k_target=3, top_p_draft=1.0,
                           top_p_target=1.0)):
        compare(wl2, gpu_step(wl2, **f), oracle_step(wl2, **f))


def test_bad_histories_give_request_statuses():
    wl = _wl("b64_g8_v152k", 4, seed=1)
    V_t = wl.target_logits.shape[1]
    hct = wl.hist_cols_t.copy()
    hct[int(wl.hist_off_t[1])] = V_t  # request 1: a column out of range
    hot = wl.hist_off_t.copy()
    wl2 = W.Workload(**{**wl.__dict__, "hist_cols_t": hct, "hist_off_t": hot})
    g = gpu_step(wl2, **QWEN25)
    o = oracle_step(wl2, **QWEN25)
    assert g["status"][1] == oracle.ST_ID_RANGE and o["status"][1] == oracle.ST_ID_RANGE
    compare(wl2, g, o)
    # a history longer than TT_MAX_HISTORY: too long
    long = np.concatenate([wl.hist_cols_t, np.zeros(3100, np.int32)])
    hot2 = wl.hist_off_t.copy()
    hot2[-1] += 3100
    wl3 = W.Workload(**{**wl.__dict__, "hist_cols_t": long, "hist_off_t": hot2})
    g = gpu_step(wl3, **QWEN25)
    assert g["status"][wl.B - 1] == 2 and np.all(g["status"][:wl.B - 1] == 0)


def test_argument_rules():
    wl = _wl("b1_g4_v32k", 1)
    inp = tt.device_inputs(wl, "cuda")
    call = lambda **f: tt.tt_step(inp["batch"], inp["vd"], inp["vt"], inp["draft_logits"],
                                  inp["target_logits"], tt.Params(**f))
    for bad in (dict(rep_penalty_target=1.1), dict(rep_penalty_draft=1.1, top_p_draft=0.9),
                dict(rep_penalty_target=1.2, top_p_target=0.9)):
        with pytest.raises(tt.TTError) as e:
            call(**bad)  # a penalty needs its family's top-k
        assert e.value.code == tt.binding.TT_ERR_UNSUPPORTED
    for bad in (dict(rep_penalty_target=0.0, top_k_target=5),
                dict(rep_penalty_draft=float("inf"), top_k_draft=5)):
        with pytest.raises(tt.TTError) as e:
            call(**bad)
        assert e.value.code == tt.binding.TT_ERR_INVALID_ARG
    hw = W.homogeneous_workload(2, 3, 500, seed=1)
    hin = tt.device_inputs(hw, "cuda")
    with pytest.raises(tt.TTError) as e:
        tt.tt_step(hin["batch"], hin["vd"], hin["vt"], hin["draft_logits"], hin["target_logits"],
                   tt.Params(full_q=True, top_k_draft=4, top_k_target=4, rep_penalty_target=1.1))
    assert e.value.code == tt.binding.TT_ERR_UNSUPPORTED


def test_transfer_and_verify_alone_with_penalties():
    wl = _wl("b64_g8_v152k", 12, seed=6)
    inp = tt.device_inputs(wl, "cuda")
    prm = inp["params"]
    for k, v in QWEN25.items():
        setattr(prm, k, v)
    al = oracle.align(wl.draft_off, wl.draft_ids, wl.target_off, wl.target_ids, wl.vd.blob,
                      wl.vd.off, wl.vt.blob, wl.vt.off, wl.spec.window)
    mp = torch.as_tensor(al["map"], dtype=torch.int32, device="cuda")
    tr = to_np(tt.tt_transfer(inp["batch"], mp, prm, draft_logits=inp["draft_logits"]))
    otr = oracle.transfer(wl.draft_off, wl.draft_cols, wl.target_off, al["map"], wl.draft_logits,
                          0.7, top_k=20, top_p=0.8, rep_penalty=1.1, hist_off=wl.hist_off_d,
                          hist_cols=wl.hist_cols_d)
    assert np.array_equal(tr["status"][:wl.B], otr["status"])
    rows = wl.draft_off[:-1].repeat(np.diff(wl.target_off)) + al["map"]
    ok = (otr["drow_bnd"][rows] & 4) == 0
    d = np.abs(tr["q_hat"][:wl.n_target] - otr["q_hat"])
    assert np.all((d[ok] <= 1e-5) & (d[ok] <= 1e-4 * otr["q_hat"][ok] + 1e-30))
    q = torch.as_tensor(otr["q_hat"], dtype=torch.float32, device="cuda")
    ve = to_np(tt.tt_verify(inp["batch"], q, inp["target_logits"], prm))
    ove = oracle.verify(wl.target_off, wl.target_cols, otr["q_hat"], wl.target_logits,
                        temp_target=0.7, seed=prm.seed, top_k_target=20, top_p_target=0.8,
                        rep_penalty_target=1.1, hist_off_t=wl.hist_off_t,
                        hist_cols_t=wl.hist_cols_t)
    g = dict(ve)
    g["q_hat"] = otr["q_hat"]
    o = dict(ove)
    o["q_hat"] = otr["q_hat"]
    compare(wl, g, o, check_align=False)


@pytest.mark.parametrize("name,n_sample", [("b64_g8_v152k", 8), ("b1024_g8_v201k_bf16", 5)])
def test_full_size_penalty_step_sampled(name, n_sample):
    wl = W.with_histories(W.make_workload(name, seed=0, device="cuda"), 64, 1024, seed=0)
    inp = tt.device_inputs(wl, "cuda")
    prm = inp["params"]
    for k, v in QWEN25.items():
        setattr(prm, k, v)
    out = to_np(tt.tt_step(inp["batch"], inp["vd"], inp["vt"], inp["draft_logits"],
                           inp["target_logits"], prm))
    m = np.diff(wl.target_off)
    assert np.all(out["status"] == 0)
    assert np.all((out["accepted"] >= 0) & (out["accepted"] <= m))
    assert np.all((out["next_token"] >= 0) & (out["next_token"] < wl.target_logits.shape[1]))
    rng = np.random.default_rng(6)
    B = wl.B
    for b in np.unique(np.concatenate([[0, B - 1], rng.choice(B, size=n_sample, replace=False)])):
        sw = sub_workload(wl, [b])
        o = oracle_step(sw, request_base=int(b), **QWEN25)
        g = dict(out)
        g["_target_off"], g["_draft_off"] = wl.target_off, wl.draft_off
        compare(sw, g, o, req_index=[b])
