"""Pins of the oracle's sampling filters (the paper's generation
hyperparameter table: temperature, top-k, top-p): hand-worked rows, the
limits where a filter does nothing or keeps one token, the tie rule, and the
speculative-sampling guarantee on filtered distributions (Alg. 4: the emitted
token is distributed as the filtered target distribution p_f whatever the
filtered draft distribution q_f is)."""
import numpy as np
import pytest
from scipy import special, stats

import oracle


def rows(p):
    return np.log(np.asarray(p, np.float64)).astype(np.float32)


def fp(z, T=1.0, k=0, p=1.0):
    return oracle.filtered_probs(np.asarray(z, np.float32)[None, :], T, k, p)


def test_hand_worked_rows():
    z = rows([0.5, 0.3, 0.15, 0.05])
    # top-p 0.79: the mass before the third token is 0.8 >= 0.79, so two tokens
    pr, lse, b = fp(z, p=0.79)
    assert np.allclose(pr, [0.625, 0.375, 0, 0], atol=1e-7) and b == 0
    assert abs(lse - np.log(0.8)) < 1e-6
    # top-p 0.81: three tokens
    pr, _, _ = fp(z, p=0.81)
    assert np.allclose(pr, [0.5 / 0.95, 0.3 / 0.95, 0.15 / 0.95, 0], atol=1e-7)
    # top-k 1: the argmax
    assert np.array_equal(fp(z, k=1)[0], [1, 0, 0, 0])
    # top-k 2 then top-p 0.5: after top-k (0.625, 0.375); the second token's
    # mass before is 0.625 >= 0.5
    assert np.allclose(fp(z, k=2, p=0.5)[0], [1, 0, 0, 0])
    # the same row at T = 0.5 squares and renormalises the probabilities
    w = np.array([0.5, 0.3, 0.15, 0.05]) ** 2
    assert np.allclose(fp(z, T=0.5)[0], w / w.sum(), atol=1e-7)


def test_ties_keep_the_smaller_column():
    z = np.array([1.0, 2.0, 2.0, 0.0], np.float32)
    assert np.array_equal(fp(z, k=1)[0], [0, 1, 0, 0])
    pr, _, _ = fp(z, k=2)
    assert pr[0] == 0 and pr[3] == 0 and abs(pr[1] - 0.5) < 1e-12 and pr[1] == pr[2]


@pytest.mark.parametrize("T", [0.6, 1.0, 1.7])
def test_limits_equal_plain_softmax(T):
    rng = np.random.default_rng(1)
    z = (rng.standard_normal(300) * 2).astype(np.float32)
    want = special.softmax(z.astype(np.float64) / T)
    for k, p in ((0, 1.0), (300, 1.0), (1000, 0.0)):
        pr, lse, _ = fp(z, T, k, p)
        assert np.allclose(pr, want, rtol=1e-12, atol=1e-15)
        assert abs(lse - special.logsumexp(z.astype(np.float64) / T)) < 1e-12
    # top-k keeps exactly k columns, the k largest
    pr, _, _ = fp(z, T, 20)
    assert np.count_nonzero(pr) == 20
    assert set(np.nonzero(pr)[0]) == set(np.argsort(-z, kind="stable")[:20])


def test_top_p_keeps_the_smallest_prefix_reaching_p():
    rng = np.random.default_rng(5)
    for _ in range(20):
        z = (rng.standard_normal(64) * 1.5).astype(np.float32)
        base = special.softmax(z.astype(np.float64))
        order = np.argsort(-z, kind="stable")
        for top_p in (0.3, 0.8, 0.95):
            pr, _, b = fp(z, 1.0, 0, top_p)
            kept = np.nonzero(pr)[0]
            n = len(kept)
            assert set(kept) == set(order[:n])
            assert base[order[:n]].sum() >= top_p - 1e-12       # reaches top_p
            assert base[order[:n - 1]].sum() < top_p + 1e-12    # and no shorter prefix does
            assert np.allclose(pr[kept], base[kept] / base[kept].sum())


def test_transfer_takes_the_filtered_draft_probability():
    zd = np.stack([rows([0.6, 0.25, 0.1, 0.05]), rows([0.1, 0.2, 0.3, 0.4])])
    # request 0: draft tokens (col 1, col 3); target positions map to draft 0, 1, 1
    r = oracle.transfer([0, 2], [1, 3], [0, 3], [0, 1, 1], zd, 1.0, top_k=2, top_p=1.0)
    assert np.allclose(r["q_hat"], [0.25 / 0.85, 0.4 / 0.7, 0.4 / 0.7])
    r = oracle.transfer([0, 2], [1, 0], [0, 1], [1], zd, 1.0, top_k=2)
    assert r["q_hat"].tolist() == [0.0]  # column 0 is outside row 1's top 2


@pytest.mark.parametrize("k,p", [(3, 1.0), (0, 0.8), (4, 0.7)])
def test_filtered_speculative_sampling_emits_the_filtered_target(k, p):
    """Draft t ~ q_f, accept with min(1, p_f/q_f), else resample the normalised
    max(0, p_f - q_f): the emitted token is distributed as p_f."""
    rng = np.random.default_rng(10 + k)
    V, N = 10, 40000
    zp = rows(rng.dirichlet(np.ones(V) * 0.8))
    zq = rows(rng.dirichlet(np.ones(V) * 0.8))
    pf = fp(zp, 1.0, k, p)[0]
    qf = fp(zq, 1.0, k, p)[0]
    t = rng.choice(V, size=N, p=qf / qf.sum())
    off = np.arange(N + 1, dtype=np.int32)
    tl = np.empty((2 * N, V), np.float32)
    tl[0::2] = zp
    tl[1::2] = zp
    dl = np.broadcast_to(zq, (N, V)).copy()
    out = oracle.verify(off, t.astype(np.int32), qf[t], tl, seed=9, full_q=True, draft_off=off,
                        mp=np.zeros(N, np.int32), draft_logits=dl, top_k_target=k,
                        top_p_target=p, top_k_draft=k, top_p_draft=p)
    first = np.where(out["accepted"] == 1, t, out["next_token"])
    counts = np.bincount(first, minlength=V)
    keep = pf > 0
    assert counts[~keep].sum() == 0
    assert stats.chisquare(counts[keep], pf[keep] * N).pvalue > 1e-4
    assert np.allclose(out["p_hat"][:5], pf[t[:5]])
