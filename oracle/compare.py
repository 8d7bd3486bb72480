"""Comparison of one verification step's device results with the oracle's
(test infrastructure, like the rest of this package: the tests, the smoke check
and the benchmark's CPU-baseline leg use it; the product path never does).

The contract it checks:
  * statuses, alignment paths, costs, maps and accepted lengths bit-exact;
  * q_hat and p_hat within 1e-5 absolute and 1e-4 relative, lse within 1e-5
    absolute (the kernels accumulate in fp32 with compensated merges);
  * a difference in a sampled quantity is excused only where the oracle's own
    arithmetic says the decision that differs lay within 1e-6 of its boundary:
      - accepted lengths that differ first disagree at position
        j = min(a_gpu, a_oracle); that decision must be a flagged boundary case
        (its uniform within 1e-6 of min(1, p/q));
      - next tokens that differ (with equal accepted lengths) must both lie in
        the closed column interval [tok_lo, tok_hi + 1] of columns whose
        running residual mass is within 1e-6 Z of the draw u' Z, which is where
        two correct inverse-CDF walks can part;
      - a row whose top-p cut lies within 1e-6 of top_p has two valid kept sets:
        its p_hat / lse (target row) or the q_hat it gives (draft row) are not
        compared, and a decision or draw is excused only if it used such a row.
Every excused case is counted; anything else is a mismatch.
"""
from __future__ import annotations

from typing import Dict, List, Optional

import numpy as np

ABS_TOL = 1e-5
REL_TOL = 1e-4
TINY = 1e-30  # below this an fp32 probability may flush to zero


def _close(g: np.ndarray, o: np.ndarray) -> np.ndarray:
    d = np.abs(np.asarray(g, np.float64) - np.asarray(o, np.float64))
    return (d <= ABS_TOL) & (d <= REL_TOL * np.abs(o) + TINY)


def compare_step(g: Dict[str, np.ndarray], o: Dict[str, np.ndarray], draft_off, target_off,
                 g_draft_off=None, g_target_off=None, req_index=None, check_align: bool = True,
                 check_q: bool = True) -> dict:
    """Compares the device outputs ``g`` (numpy arrays of the whole device batch)
    with the oracle outputs ``o`` (for the requests it ran). ``draft_off`` /
    ``target_off`` are the oracle batch's CSR offsets, ``g_*_off`` the device
    batch's (default: the same), and ``req_index[b]`` the device request that
    oracle request b is. Returns counts of the excused cases and a list of
    mismatches (empty when the two agree under the contract)."""
    draft_off = np.asarray(draft_off)
    target_off = np.asarray(target_off)
    g_draft_off = draft_off if g_draft_off is None else np.asarray(g_draft_off)
    g_target_off = target_off if g_target_off is None else np.asarray(g_target_off)
    B = len(o["status"])
    gi = np.arange(B) if req_index is None else np.asarray(req_index)
    row_bnd = o.get("row_bnd")
    drow_bnd = o.get("drow_bnd")
    tok_lo, tok_hi = o.get("tok_lo"), o.get("tok_hi")
    bad: List[str] = []
    n_acc = n_tok = n_filt = 0
    for b in range(B):
        gb = int(gi[b])
        if int(g["status"][gb]) != int(o["status"][b]):
            bad.append("request %d: status %d != %d" % (b, g["status"][gb], o["status"][b]))
            continue
        if o["status"][b] != 0:
            if g["accepted"][gb] != 0 or g["next_token"][gb] != -1:
                bad.append("request %d: failed request with outputs" % b)
            continue
        ot0, ot1 = int(target_off[b]), int(target_off[b + 1])
        gt0, gt1 = int(g_target_off[gb]), int(g_target_off[gb + 1])
        od0 = int(draft_off[b])
        m = ot1 - ot0
        omap = o["map"][ot0:ot1] if "map" in o else None
        if check_align and "path_len" in g:
            L = int(o["path_len"][b])
            op = od0 + ot0
            gp = int(g_draft_off[gb]) + gt0
            if int(g["path_len"][gb]) != L or int(g["cost"][gb]) != int(o["cost"][b]):
                bad.append("request %d: path length or cost" % b)
                continue
            if not np.array_equal(g["path"][2 * gp:2 * (gp + L)], o["path"][op:op + L].ravel()):
                bad.append("request %d: path" % b)
                continue
            if not np.array_equal(g["map"][gt0:gt1], omap):
                bad.append("request %d: map" % b)
                continue
        # rows with an ambiguous kept set (target rows 0..m, mapped draft rows)
        rb = (np.zeros(m + 1, np.int32) if row_bnd is None
              else np.asarray(row_bnd[ot0 + b:ot1 + b + 1]))
        t_amb = (rb & 4) != 0
        q_amb = np.zeros(m, bool)
        if drow_bnd is not None and omap is not None and len(drow_bnd):
            q_amb = (np.asarray(drow_bnd)[od0 + omap] & 4) != 0
        pos_amb = t_amb[:m] | q_amb  # position j's decision used an ambiguous row
        if check_q and "q_hat" in g:
            ok = _close(g["q_hat"][gt0:gt1], o["q_hat"][ot0:ot1]) | q_amb
            if not ok.all():
                bad.append("request %d: q_hat at %s" % (b, np.nonzero(~ok)[0].tolist()))
        ok = _close(g["p_hat"][gt0:gt1], o["p_hat"][ot0:ot1]) | t_amb[:m]
        if not ok.all():
            bad.append("request %d: p_hat at %s" % (b, np.nonzero(~ok)[0].tolist()))
        if "lse" in g:
            gl = np.asarray(g["lse"][gt0 + gb:gt1 + gb + 1], np.float64)
            ol = np.asarray(o["lse"][ot0 + b:ot1 + b + 1], np.float64)
            ok = (np.abs(gl - ol) <= ABS_TOL) | t_amb
            if not ok.all():
                bad.append("request %d: lse at rows %s" % (b, np.nonzero(~ok)[0].tolist()))
        ag, ao = int(g["accepted"][gb]), int(o["accepted"][b])
        if ag != ao:
            j = min(ag, ao)  # the first decision the two disagree on
            if j < m and rb[j] & 1:
                n_acc += 1
            elif j < m and pos_amb[j]:
                n_filt += 1
            else:
                bad.append("request %d: accepted %d != %d (decision %d not a boundary case)"
                           % (b, ag, ao, j))
            continue
        tg, to = int(g["next_token"][gb]), int(o["next_token"][b])
        if tg != to:
            a = ao
            lo = -1 if tok_lo is None else int(tok_lo[b])
            hi = -1 if tok_hi is None else int(tok_hi[b])
            row_amb = bool(t_amb[a] or (rb[a] & 8) or (a < m and q_amb[a]))
            if lo >= 0 and lo <= min(tg, to) and max(tg, to) <= hi + 1:
                n_tok += 1
            elif row_amb:
                n_filt += 1
            else:
                bad.append("request %d: next token %d != %d (boundary columns %d..%d)"
                           % (b, tg, to, lo, hi))
    return dict(requests=B, accept_boundary=n_acc, token_boundary=n_tok, filter_boundary=n_filt,
                mismatches=bad)
