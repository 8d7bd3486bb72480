"""Comparison of the CUDA path (through the C ABI) with the CPU oracle on the
same seeded inputs. Tolerances follow the method's contract: alignment paths,
costs, maps, statuses and accepted lengths bit-exact; probabilities within
1e-5 absolute and 1e-4 relative, log-normalisers within 1e-5 absolute (fp32
accumulation); sampled tokens equal except at the one decision where the
oracle's uniform lay within 1e-6 of its boundary (those cases are counted,
never hidden)."""
from __future__ import annotations

import numpy as np
import torch

import oracle
import paper_2510_15545_gb300 as tt
from oracle.compare import compare_step
from paper_2510_15545_gb300 import workload as W

TOL = 1e-5  # absolute bound on probabilities


def to_np(out: dict) -> dict:
    return {k: v.detach().cpu().numpy() for k, v in out.items()}


def gpu_step(wl, *, device="cuda", window=None, temp_draft=None, temp_target=None, seed=None,
             full_q=False, draft_probs=None, request_base=0, top_k_draft=0, top_p_draft=1.0,
             top_k_target=0, top_p_target=1.0, rep_penalty_draft=1.0,
             rep_penalty_target=1.0) -> dict:
    inp = tt.device_inputs(wl, device)
    prm = inp["params"]
    prm.top_k_draft, prm.top_p_draft = top_k_draft, top_p_draft
    prm.top_k_target, prm.top_p_target = top_k_target, top_p_target
    prm.rep_penalty_draft, prm.rep_penalty_target = rep_penalty_draft, rep_penalty_target
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
    """Asserts parity of one step (the contract of ``oracle.compare``: exact
    integers, 1e-5 absolute and 1e-4 relative probabilities, a sampled result
    excused only at the decision the oracle flags as a boundary case); returns
    the counts of excused cases. ``req_index[b]`` maps the oracle's request b to
    the GPU's (sampled runs)."""
    r = compare_step(g, o, wl.draft_off, wl.target_off, g_draft_off=g.get("_draft_off"),
                     g_target_off=g.get("_target_off"), req_index=req_index,
                     check_align=check_align, check_q=check_q)
    assert not r["mismatches"], r["mismatches"][:8]
    return r
