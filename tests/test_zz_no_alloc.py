"""tt_step_noalloc, the verification step for callers that cannot allocate
device memory (their runtime owns all device memory, their serving loop must
not stall on the allocator, or they only hand over inputs and outputs). It
uses the library's own fixed scratch instead of a caller's workspace; here it
is called through the C ABI and checked against tt_step on the same inputs,
on two calls in a row (each call finds the scratch as the one before left it).
This file is collected last so that a run stopping at the first failure has
already run every other test."""
import ctypes

import numpy as np
import pytest
import torch

import paper_2510_15545_gb300 as tt
from paper_2510_15545_gb300 import binding
from paper_2510_15545_gb300 import workload as W

TOL = 1e-5
_CACHE = {}


def test_batch_beyond_the_scratch_is_refused_on_the_host():
    # 10 million target tokens need far more than the 16 MiB scratch: refused
    # before anything touches the GPU (no pointer below is ever dereferenced)
    lib = tt.load(build_if_missing=True)
    b = binding._Batch(1, 1, 10_000_000, 1, 1, 16, 16, None, 16, 16, None)
    v = binding._Vocab(16, 16, 1, 1)
    lg = binding._Logits(256, binding.TT_F32, 151936, 151936, 10_000_001)
    out = binding._StepOut(16, 16, 16, None, None, None, None, None, None, None)
    keep = []
    code = lib.tt_step_noalloc(ctypes.byref(b), ctypes.byref(v), ctypes.byref(v),
                               ctypes.byref(lg), None, ctypes.byref(lg),
                               ctypes.byref(binding.Params()._c(keep)), ctypes.byref(out), None)
    assert code == binding.TT_ERR_UNSUPPORTED


def test_invalid_params_are_refused_before_the_size_check():
    # an invalid top-k (-1) must not slip past the size check: tt_step's own
    # checks run first and refuse the call before anything touches the GPU
    lib = tt.load(build_if_missing=True)
    b = binding._Batch(1, 1, 10_000_000, 1, 1, 16, 16, None, 16, 16, None)
    v = binding._Vocab(16, 16, 1, 1)
    lg = binding._Logits(256, binding.TT_F32, 151936, 151936, 10_000_001)
    out = binding._StepOut(16, 16, 16, None, None, None, None, None, None, None)
    keep = []
    for bad in (dict(top_k_target=-1), dict(top_k_draft=-1), dict(top_k_target=33),
                dict(temp_target=0.0)):
        prm = binding.Params(**bad)._c(keep)
        code = lib.tt_step_noalloc(ctypes.byref(b), ctypes.byref(v), ctypes.byref(v),
                                   ctypes.byref(lg), None, ctypes.byref(lg), ctypes.byref(prm),
                                   ctypes.byref(out), None)
        assert code == binding.TT_ERR_INVALID_ARG, bad


def _check_same(wl, ref, got):
    for k in ("status", "accepted", "next_token", "path_len", "cost", "map"):
        assert torch.equal(ref[k], got[k]), k
    for k in ("q_hat", "p_hat", "lse"):
        assert float((ref[k] - got[k]).abs().max()) <= TOL, k
    path_r, path_g = ref["path"].cpu(), got["path"].cpu()
    for b in range(wl.B):
        p0 = int(wl.draft_off[b] + wl.target_off[b])
        L = int(ref["path_len"][b])
        assert torch.equal(path_r[2 * p0:2 * (p0 + L)], path_g[2 * p0:2 * (p0 + L)])


@pytest.mark.gpu
def test_noalloc_step_equals_step_on_two_calls_in_a_row():
    if not torch.cuda.is_available():
        pytest.skip("needs a GPU")
    tt.load(build_if_missing=True)
    workloads = [W.make_workload("b64_g8_v152k", B=16, seed=3, vocab_cache=_CACHE),
                 W.make_workload("b1024_g8_v201k_bf16", B=8, seed=4, vocab_cache=_CACHE),
                 W.make_workload("dtw_4096x64", B=24, seed=5, vocab_cache=_CACHE)]
    filters = dict(temp_draft=0.7, temp_target=0.7, top_k_draft=20, top_p_draft=0.8,
                   top_k_target=20, top_p_target=0.8)
    cases = [(wl, {}, False) for wl in workloads]
    cases.append((workloads[0], filters, False))  # kept sets and lists in the scratch
    cases.append((workloads[1], {}, True))        # caller-given draft probabilities
    for wl, f, given in cases:
        inp = tt.device_inputs(wl, "cuda")
        prm = inp["params"]
        for k, v in f.items():
            setattr(prm, k, v)
        probs = None
        if given:
            probs = torch.rand(wl.n_draft, device="cuda") * 0.9 + 0.05
        args = (inp["batch"], inp["vd"], inp["vt"], inp["draft_logits"], inp["target_logits"],
                prm)
        ref = tt.tt_step(*args, draft_probs=probs)
        first = tt.tt_step_noalloc(*args, draft_probs=probs)
        second = tt.tt_step_noalloc(*args, draft_probs=probs)
        torch.cuda.synchronize()
        assert int((ref["status"] != 0).sum()) == 0
        _check_same(wl, ref, first)
        _check_same(wl, ref, second)
