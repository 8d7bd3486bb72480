"""Comparison of the CUDA path (through the C ABI) with the CPU oracle on the
same seeded inputs. Tolerances follow the method's contract: alignment paths,
costs, maps, statuses and accepted lengths bit-exact; probabilities and
log-normalisers within 1e-5 absolute (fp32 accumulation); sampled tokens equal
except where the oracle's uniform lay within 1e-6 of a decision boundary (those
cases are counted, never hidden)."""
from __future__ import annotations

import numpy as np
import torch

import oracle
import paper_2510_15545_gb300 as tt
from paper_2510_15545_gb300 import workload as W

TOL = 1e-5


def to_np(out: dict) -> dict:
    return {k: v.detach().cpu().numpy() for k, v in out.items()}


def gpu_step(wl, *, device="cuda", window=None, temp_draft=None, temp_target=None, seed=None,
             full_q=False, draft_probs=None, request_base=0, top_k_draft=0, top_p_draft=1.0,
             top_k_target=0, top_p_target=1.0) -> dict:
    inp = tt.device_inputs(wl, device)
    prm = inp["params"]
    prm.top_k_draft, prm.top_p_draft = top_k_draft, top_p_draft
    prm.top_k_target, prm.top_p_target = top_k_target, top_p_target
    if window is not None:
        prm.window = window
    if temp_draft is not None:
        prm.temp_draft = temp_draft
    if temp_target is not None:
        prm.temp_target = temp_target
    if seed is not None:
        prm.seed = seed
    prm.full_q = full_q
    prm.request_base = request_base
    probs = None if draft_probs is None else torch.as_tensor(draft_probs, dtype=torch.float32,
                                                             device=device)
    out = tt.tt_step(inp["batch"], inp["vd"], inp["vt"], inp["draft_logits"],
                     inp["target_logits"], prm, draft_probs=probs)
    torch.cuda.synchronize()
    return to_np(out)


def oracle_step(wl, **kw) -> dict:
    return oracle.step(wl, **kw)


def sub_workload(wl, idx) -> W.Workload:
    """Requests ``idx`` of a workload as a workload of their own (logits on the CPU)."""
    return wl.subset(idx)


def compare(wl, g: dict, o: dict, req_index=None, check_align=True, check_q=True) -> dict:
    """Asserts parity of one step; returns counts of boundary cases.
    ``req_index[b]`` maps the oracle's request b to the GPU's (sampled runs)."""
    B = len(o["status"])
    gi = np.arange(B) if req_index is None else np.asarray(req_index)
    g_off_t = g.get("_target_off", wl.target_off)
    g_off_d = g.get("_draft_off", wl.draft_off)
    assert np.array_equal(g["status"][gi], o["status"]), (g["status"][gi], o["status"])
    n_acc_b = n_tok_b = n_filt_b = 0
    for b in range(B):
        if o["status"][b] != 0:
            assert g["accepted"][gi[b]] == 0 and g["next_token"][gi[b]] == -1
            continue
        gb = gi[b]
        ot0, ot1 = int(wl.target_off[b]), int(wl.target_off[b + 1])
        gt0, gt1 = int(g_off_t[gb]), int(g_off_t[gb + 1])
        if check_align and "path_len" in g:
            L = int(o["path_len"][b])
            assert int(g["path_len"][gb]) == L, b
            assert int(g["cost"][gb]) == int(o["cost"][b]), b
            op = int(wl.draft_off[b]) + ot0
            gp = int(g_off_d[gb]) + gt0
            assert np.array_equal(g["path"][2 * gp:2 * (gp + L)], o["path"][op:op + L].ravel()), b
            assert np.array_equal(g["map"][gt0:gt1], o["map"][ot0:ot1]), b
        if int(o["boundary"][b]) & 4:
            # a top-p cut within 1e-6 of the mass before some token: the kept
            # sets may differ, so nothing downstream is compared
            n_filt_b += 1
            continue
        if check_q and "q_hat" in g:
            assert np.max(np.abs(g["q_hat"][gt0:gt1] - o["q_hat"][ot0:ot1]), initial=0) <= TOL, b
        assert np.max(np.abs(g["p_hat"][gt0:gt1] - o["p_hat"][ot0:ot1]), initial=0) <= TOL, b
        if "lse" in g:
            gl = g["lse"][gt0 + gb:gt1 + gb + 1]
            ol = o["lse"][ot0 + b:ot1 + b + 1]
            assert np.max(np.abs(gl - ol)) <= TOL * max(1.0, float(np.max(np.abs(ol)))), b
        bnd = int(o["boundary"][b])
        if g["accepted"][gb] != o["accepted"][b]:
            assert bnd & 1, (b, g["accepted"][gb], o["accepted"][b])
            n_acc_b += 1
            continue
        if g["next_token"][gb] != o["next_token"][b]:
            assert bnd & 2, (b, g["next_token"][gb], o["next_token"][b])
            n_tok_b += 1
    return dict(requests=B, accept_boundary=n_acc_b, token_boundary=n_tok_b,
                filter_boundary=n_filt_b)
