"""Which way the nucleus kernels settle each row in the GPU nucleus tests,
computed on the CPU from the same seeded inputs. Rows of at most 8192 columns
take one warp each: the columns within 12 log2 units of the row maximum (at
most 512) are the candidates. Wider rows take one CTA each: the columns within
14 log2 units, at most 512 in each of the CTA's eight warp regions (vector v
of a row goes to thread v mod 256). Either way the cut must lie among the
candidates and its 1/32-log2-unit bucket hold at most 32 (warp) or 256 (CTA)
of them; other rows take the full histogram levels. The paper's settings
(App. F: T 0.6 with top-p 0.9 or 0.95) take the candidate ways on every
workload; rows of coarse integer logits take the histogram levels and rows
with one dominant logit a single candidate, so the GPU tests cover both."""
import dataclasses
import os

import numpy as np
import torch

from paper_2510_15545_gb300 import workload as W

LOG2E = 1.4426950408889634


def _candidate_way(logits: torch.Tensor, T: float, p: float) -> np.ndarray:
    """Per row: True when the candidate way (warp or CTA) settles it."""
    V = logits.shape[1]
    narrow = V <= 8192
    D, cross_cap = (12.0, 32) if narrow else (14.0, 256)
    vec = 4 if logits.dtype == torch.float32 else 8
    nvec = V // vec
    z = logits.float().numpy().astype(np.float64) * (LOG2E / T)
    d = z.max(1, keepdims=True) - z
    total = np.exp2(-d).sum(1)
    out = np.zeros(len(d), bool)
    for r in range(len(d)):
        cols = np.nonzero(d[r] < D)[0]
        if narrow:
            if len(cols) > 512:
                continue
        else:
            v = cols // vec
            tid = np.where(cols < nvec * vec, v % 256, (cols - nvec * vec) % 256)
            if np.bincount(tid // 32, minlength=8).max() > 512:
                continue
        dc = d[r][cols]
        order = np.lexsort((cols, dc))  # larger logit first, then smaller column
        mc = np.exp2(-dc[order])
        before = np.cumsum(mc) - mc
        kept = before < p * total[r]
        if kept.all() and mc.sum() < p * total[r]:
            continue  # the cut lies beyond the candidates
        last = dc[order][kept.sum() - 1]
        if last > D - 0.5:
            continue  # too near the candidates' edge to claim either way
        same = np.floor(dc * 32) == np.floor(last * 32)
        out[r] = same.sum() <= cross_cap - 4
    return out


def test_the_table_settings_take_the_candidate_ways():
    for name, B in (("b64_g8_v152k", 12), ("b1024_g8_v201k_bf16", 8),
                    ("b256_g16_v152k_bf16", 4), ("dtw_4096x64", 6), ("b1_g4_v32k", 1)):
        wl = W.make_workload(name, B=B, seed=3)
        for p in (0.9, 0.95):
            for L in (wl.target_logits, wl.draft_logits):
                assert _candidate_way(L, 0.6, p).all(), (name, p)


def test_coarse_integer_rows_take_the_histogram_levels():
    wl = W.make_workload("b64_g8_v152k", B=8, seed=11)
    rng = np.random.default_rng(5)
    tl = torch.as_tensor(rng.integers(-3, 4, size=wl.target_logits.shape).astype(np.float32))
    tl[::3, 17] = 60.0
    wl2 = dataclasses.replace(wl, target_logits=tl)
    way = _candidate_way(wl2.target_logits, 0.6, 0.9)
    dominant = np.zeros(len(way), bool)
    dominant[::3] = True
    assert way[dominant].all() and not way[~dominant].any()


def test_crowded_rows_take_the_second_candidate_pass():
    """The rows of test_gpu_nucleus.crowded_rows: more than 4096 candidates
    within 14 log2 units, so the first pass overflows; the count below each
    whole bar (the kernel estimates it from the candidates it holds) gives the
    largest bar with at most 3200, and the second pass at that bar holds the
    cut with every warp's candidates within its region."""
    import sys
    sys.path.insert(0, os.path.dirname(os.path.abspath(__file__)))
    import importlib
    gn = importlib.import_module("test_gpu_nucleus")
    wl = gn.crowded_rows(W.make_workload("b64_g8_v152k", B=6, seed=13))
    z = wl.target_logits.numpy().astype(np.float64) * (LOG2E / 0.6)
    d = z.max(1, keepdims=True) - z
    m = np.exp2(-d)
    V = d.shape[1]
    for r in range(len(d)):
        assert (d[r] < 14).sum() > 4096                     # the first pass overflows
        bar = max(b for b in range(8, 14) if (d[r] < b).sum() <= 3200)
        cols = np.nonzero(d[r] < bar)[0]
        tid = (cols // 4) % 256                              # fp32: 4 columns per vector
        assert np.bincount(tid // 32, minlength=8).max() <= 512
        assert m[r][cols].sum() >= 0.5 * m[r].sum()          # the cut lies below the bar
        assert V > 8192                                      # the CTA kernel's rows
