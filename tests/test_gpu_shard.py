"""GPU parity of the vocabulary-sharded verification (tt_verify_sharded):
target rows split by columns into S separate logits arrays, each reduced on
its own, the per-shard records merged (split-lse) and the residual drawn by
shard, chunk and column. The result must be the verification of the whole rows
(the oracle, and tt_verify on the unsplit rows), whatever the split: one
shard, even and ragged widths, a shard of one column holding a scored token,
eight shards, fp32 and bf16 rows, other temperatures and seeds."""
import numpy as np
import pytest
import torch

import oracle
import paper_2510_15545_gb300 as tt
from paper_2510_15545_gb300 import workload as W
from _parity import compare, to_np

pytestmark = pytest.mark.gpu
_CACHE = {}


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.skip("needs a GPU")
    tt.load(build_if_missing=True)


def _split(t: torch.Tensor, widths):
    """Column slices of t as separate GPU tensors, rows padded to 16 bytes plus
    one more 16-byte vector of NaN (a read past a slice shows)."""
    per16 = 16 // t.element_size()
    out, c = [], 0
    for w in widths:
        buf = torch.full((t.shape[0], (w + per16 - 1) // per16 * per16 + per16), float("nan"),
                         dtype=t.dtype, device="cuda")
        buf[:, :w] = t[:, c:c + w].to("cuda")
        out.append(buf[:, :w])
        c += w
    assert c == t.shape[1]
    return out


def _widths(V, cuts):
    edges = [0] + sorted(cuts) + [V]
    return [b - a for a, b in zip(edges, edges[1:])]


def _run(wl, widths, temp=1.0, seed=None):
    inp = tt.device_inputs(wl, "cuda")
    prm = inp["params"]
    prm.temp_target = temp
    if seed is not None:
        prm.seed = seed
    al = oracle.align(wl.draft_off, wl.draft_ids, wl.target_off, wl.target_ids, wl.vd.blob,
                      wl.vd.off, wl.vt.blob, wl.vt.off, wl.spec.window)
    otr = oracle.transfer(wl.draft_off, wl.draft_cols, wl.target_off, al["map"], wl.draft_logits,
                          prm.temp_draft)
    q = torch.as_tensor(otr["q_hat"], dtype=torch.float32, device="cuda")
    g = to_np(tt.tt_verify_sharded(inp["batch"], q, _split(wl.target_logits, widths), prm,
                                   summaries=True))
    o = oracle.verify(wl.target_off, wl.target_cols, otr["q_hat"], wl.target_logits,
                      temp_target=temp, seed=prm.seed)
    gg, oo = dict(g), dict(o)
    gg["q_hat"] = oo["q_hat"] = otr["q_hat"]
    r = compare(wl, gg, oo, check_align=False)
    # the unsplit rows through tt_verify meet the same bar
    u = to_np(tt.tt_verify(inp["batch"], q, inp["target_logits"], prm))
    uu = dict(u)
    uu["q_hat"] = otr["q_hat"]
    compare(wl, uu, oo, check_align=False)
    assert np.array_equal(u["status"], g["status"])
    assert np.max(np.abs(u["p_hat"] - g["p_hat"])) <= 1e-5
    return g, o, r


def _check_records(wl, g, widths):
    """Exactly one shard owns each scored column of a verified position (its
    record carries the scored logit), none on a bonus row."""
    rec = g["summaries"]
    owned = ~np.isnan(rec[:, :, 3])
    for b in range(wl.B):
        t0, t1 = int(wl.target_off[b]), int(wl.target_off[b + 1])
        for j in range(t1 - t0 + 1):
            row = t0 + b + j
            n = int(owned[:, row].sum())
            if j < t1 - t0:
                col = int(wl.target_cols[t0 + j])
                k = int(np.searchsorted(np.cumsum(widths), col, side="right"))
                assert n == 1 and owned[k, row], (b, j)
            else:
                assert n == 0, (b, j)


@pytest.mark.parametrize("cuts", [[], [75968], [1000, 51000], [1, 2048, 4097, 30000, 60000,
                                                                 90000, 120000]])
def test_fp32_rows_split_every_way(cuts):
    wl = W.make_workload("b64_g8_v152k", B=16, seed=7, vocab_cache=_CACHE)
    widths = _widths(wl.target_logits.shape[1], cuts)
    g, o, r = _run(wl, widths)
    _check_records(wl, g, widths)
    assert r["token_boundary"] <= 2


@pytest.mark.parametrize("temp,seed", [(1.0, None), (0.6, 99)])
def test_bf16_rows_in_four_ragged_shards(temp, seed):
    wl = W.make_workload("b1024_g8_v201k_bf16", B=12, seed=8, vocab_cache=_CACHE)
    widths = _widths(wl.target_logits.shape[1], [333, 70001, 150000])
    g, o, r = _run(wl, widths, temp=temp, seed=seed)
    _check_records(wl, g, widths)


def test_scored_column_alone_in_a_shard():
    wl = W.homogeneous_workload(24, 5, 3000, seed=11)
    t = int(wl.target_cols[0])
    cuts = sorted({t, t + 1} - {0, 3000})
    widths = _widths(3000, cuts)
    g, o, r = _run(wl, widths)
    _check_records(wl, g, widths)


def test_many_requests_match_unsplit_verify():
    # 256 homogeneous requests, frequent acceptance and residual draws across
    # all eight shards
    wl = W.homogeneous_workload(256, 6, 20000, seed=12)
    widths = _widths(20000, [2500 * i for i in range(1, 8)])
    g, o, r = _run(wl, widths, temp=0.8)
    assert r["requests"] == 256
