"""GPU parity of the sampling filters (temperature, top-k, top-p; the paper's
generation hyperparameter table) against the oracle, through the C ABI
(top-p without top-k in test_gpu_nucleus.py):
tt_step in one-hot and full-q mode, tt_transfer and tt_verify alone, rows with
many equal logits (the exact fallback of the candidate selection), and the
argument rules."""
import numpy as np
import pytest
import torch

import oracle
import paper_2510_15545_gb300 as tt
from paper_2510_15545_gb300 import workload as W
from _parity import compare, gpu_step, to_np

pytestmark = pytest.mark.gpu
_CACHE = {}


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.skip("needs a GPU")
    tt.load(build_if_missing=True)


def _wl(name, B, seed=0):
    return W.make_workload(name, B=B, seed=seed, vocab_cache=_CACHE)


FILTERS = [
    dict(top_k_draft=20, top_p_draft=0.95, top_k_target=20, top_p_target=0.95),  # Qwen3-32B
    dict(top_k_draft=20, top_p_draft=0.8, top_k_target=20, top_p_target=0.8),    # Qwen2.5-0.5B
    dict(top_k_draft=20, top_p_draft=1.0),                                        # draft only
    dict(top_k_target=20, top_p_target=0.9),                                      # target only
    dict(top_k_draft=1, top_k_target=1),                                          # greedy
    dict(top_k_draft=32, top_p_draft=0.5, top_k_target=5, top_p_target=1.0),
]


@pytest.mark.parametrize("f", FILTERS)
@pytest.mark.parametrize("name,B", [("b64_g8_v152k", 12), ("b1024_g8_v201k_bf16", 12)])
def test_step_with_filters_matches_oracle(f, name, B):
    wl = _wl(name, B, seed=3)
    kw = dict(temp_draft=0.6, temp_target=0.6)
    g = gpu_step(wl, **kw, **f)
    o = oracle.step(wl, **kw, **f)
    r = compare(wl, g, o)
    assert r["filter_boundary"] <= B // 4, r


@pytest.mark.parametrize("f", [FILTERS[0], dict(top_k_draft=3, top_k_target=3),
                               dict(top_k_draft=32, top_p_draft=0.7, top_k_target=32,
                                    top_p_target=0.7)])
def test_full_q_step_with_filters_matches_oracle(f):
    wl = W.homogeneous_workload(48, 6, 3000, seed=4)
    g = gpu_step(wl, full_q=True, temp_draft=0.7, temp_target=0.7, **f)
    o = oracle.step(wl, full_q=True, temp_draft=0.7, temp_target=0.7, **f)
    compare(wl, g, o)


def _tied_workload(seed):
    """Logits on a coarse integer grid: many equal logits per chunk, so the
    chunk selection meets more candidates than its shared buffer holds."""
    wl = W.homogeneous_workload(16, 4, 9000, seed=seed)
    dl = torch.round(wl.draft_logits * 0.6).float()
    tl = torch.round(wl.target_logits * 0.6).float()
    return W.Workload(spec=wl.spec, vd=wl.vd, vt=wl.vt, draft_off=wl.draft_off,
                      draft_ids=wl.draft_ids, target_off=wl.target_off,
                      target_ids=wl.target_ids, draft_cols=wl.draft_cols,
                      target_cols=wl.target_cols, draft_logits=dl, target_logits=tl)


@pytest.mark.parametrize("k,p", [(20, 1.0), (32, 0.9), (7, 0.6)])
def test_ties_and_candidate_overflow(k, p):
    wl = _tied_workload(k)
    f = dict(top_k_draft=k, top_p_draft=p, top_k_target=k, top_p_target=p)
    for full_q in (False, True):
        g = gpu_step(wl, full_q=full_q, **f)
        o = oracle.step(wl, full_q=full_q, **f)
        compare(wl, g, o)


def _padded(t: torch.Tensor) -> torch.Tensor:
    """``t`` on the GPU as a view into rows padded to a 16-byte multiple plus
    one more 16-byte vector, the padding NaN: a read past a row's end shows."""
    R, V = t.shape
    per16 = 16 // t.element_size()
    buf = torch.full((R, (V + per16 - 1) // per16 * per16 + per16), float("nan"),
                     dtype=t.dtype, device="cuda")
    buf[:, :V] = t.to("cuda")
    return buf[:, :V]


# (V, dtype, k): a unit with a ragged tail only (4100 bf16, 2053 fp32), fewer
# lanes' worth of columns than k (threshold -inf: 100 fp32 ranked, 150 bf16
# past the candidate buffer), one short unit (37 bf16), several units (6001 bf16)
@pytest.mark.parametrize("V,dtype,k", [(37, torch.bfloat16, 20), (150, torch.bfloat16, 20),
                                       (100, torch.float32, 20), (4100, torch.bfloat16, 20),
                                       (2053, torch.float32, 32), (6001, torch.bfloat16, 7)])
def test_narrow_and_ragged_rows(V, dtype, k):
    wl = W.homogeneous_workload(6, 4, V, seed=V, dtype=dtype)
    f = dict(top_k_draft=k, top_p_draft=0.9, top_k_target=k, top_p_target=0.9)
    inp = tt.device_inputs(wl, "cuda")
    dl, tl = _padded(wl.draft_logits), _padded(wl.target_logits)
    for full_q in (False, True):
        prm = inp["params"]
        prm.temp_draft = prm.temp_target = 0.8
        prm.full_q = full_q
        prm.top_k_draft, prm.top_p_draft = k, 0.9
        prm.top_k_target, prm.top_p_target = k, 0.9
        g = to_np(tt.tt_step(inp["batch"], inp["vd"], inp["vt"], dl, tl, prm))
        o = oracle.step(wl, full_q=full_q, temp_draft=0.8, temp_target=0.8, **f)
        compare(wl, g, o)


def test_transfer_and_verify_alone_with_filters():
    wl = _wl("b64_g8_v152k", 16, seed=5)
    inp = tt.device_inputs(wl, "cuda")
    prm = inp["params"]
    prm.temp_draft = prm.temp_target = 0.6
    prm.top_k_draft, prm.top_p_draft = 20, 0.95
    prm.top_k_target, prm.top_p_target = 12, 0.85
    al = oracle.align(wl.draft_off, wl.draft_ids, wl.target_off, wl.target_ids, wl.vd.blob,
                      wl.vd.off, wl.vt.blob, wl.vt.off, wl.spec.window)
    mp = torch.as_tensor(al["map"], dtype=torch.int32, device="cuda")
    tr = to_np(tt.tt_transfer(inp["batch"], mp, prm, draft_logits=inp["draft_logits"]))
    otr = oracle.transfer(wl.draft_off, wl.draft_cols, wl.target_off, al["map"], wl.draft_logits,
                          0.6, top_k=20, top_p=0.95)
    assert np.array_equal(tr["status"][:wl.B], otr["status"])
    ok = otr["boundary"] == 0
    for b in np.nonzero(ok)[0]:
        t0, t1 = wl.target_off[b], wl.target_off[b + 1]
        assert np.max(np.abs(tr["q_hat"][t0:t1] - otr["q_hat"][t0:t1])) <= 1e-5
    q = torch.as_tensor(otr["q_hat"], dtype=torch.float32, device="cuda")
    ve = to_np(tt.tt_verify(inp["batch"], q, inp["target_logits"], prm))
    ove = oracle.verify(wl.target_off, wl.target_cols, otr["q_hat"], wl.target_logits,
                        temp_target=0.6, seed=prm.seed, top_k_target=12, top_p_target=0.85)
    g = dict(ve)
    g["q_hat"] = otr["q_hat"]
    o = dict(ove)
    o["q_hat"] = otr["q_hat"]
    compare(wl, g, o, check_align=False)


def test_filter_argument_rules():
    wl = _wl("b1_g4_v32k", 1)
    inp = tt.device_inputs(wl, "cuda")
    call = lambda **f: tt.tt_step(inp["batch"], inp["vd"], inp["vt"], inp["draft_logits"],
                                  inp["target_logits"], tt.Params(**f))
    with pytest.raises(tt.TTError) as e:
        call(top_k_target=33)
    assert e.value.code == tt.binding.TT_ERR_INVALID_ARG
    with pytest.raises(tt.TTError) as e:
        call(top_k_target=4, top_p_target=0.0)
    assert e.value.code == tt.binding.TT_ERR_INVALID_ARG
    hw = W.homogeneous_workload(2, 3, 500, seed=1)
    hin = tt.device_inputs(hw, "cuda")
    with pytest.raises(tt.TTError) as e:
        tt.tt_step(hin["batch"], hin["vd"], hin["vt"], hin["draft_logits"], hin["target_logits"],
                   tt.Params(full_q=True, top_k_target=4))
    assert e.value.code == tt.binding.TT_ERR_UNSUPPORTED
    # full-q has no nucleus rows (top-p without top-k): one-hot transfer only
    with pytest.raises(tt.TTError) as e:
        tt.tt_step(hin["batch"], hin["vd"], hin["vt"], hin["draft_logits"], hin["target_logits"],
                   tt.Params(full_q=True, top_p_draft=0.9, top_p_target=0.9))
    assert e.value.code == tt.binding.TT_ERR_UNSUPPORTED
