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


def _np_uniform(seed, pos, stream, req):
    # numpy's own Philox4x64-10 at counter (pos, stream, req, 0), key (seed, 0)
    mask = (1 << 64) - 1
    c = (pos + (stream << 64) + (req << 128) - 1) & ((1 << 256) - 1)
    words = np.array([(c >> (64 * i)) & mask for i in range(4)], dtype=np.uint64)
    g = np.random.Philox(key=np.array([seed, 0], dtype=np.uint64), counter=words)
    return (int(g.random_raw(1)[0]) >> 40) / 2.0**24


def _kept_by_hand(z, T, k, p):
    """Temperature, the k largest logits (ties: smaller column), softmax over
    them, the smallest prefix whose mass reaches p, renormalised (R22-R24)."""
    s = z.astype(np.float64) / T
    order = np.argsort(-z, kind="stable")[:k]
    w = np.exp(s[order] - s[order].max())
    w /= w.sum()
    n = 0
    before = 0.0
    while n < len(order) and before < p:
        before += w[n]
        n += 1
    out = np.zeros(len(z))
    out[order[:n]] = w[:n] / w[:n].sum()
    return out


def test_filtered_decisions_recomputed_by_hand():
    """Every accept decision and next token of a filtered verification: p_f
    from the kept set built by hand, accept while u_j < p_f(t_j) / q_j, the
    residual (p_f with t_a's mass lowered by q_hat, zero outside the kept set,
    or the bonus row's p_f) sampled in column order (R27)."""
    rng = np.random.default_rng(33)
    B, V, seed, T, k, p = 300, 40, 5, 0.7, 6, 0.9
    ms = rng.integers(1, 5, size=B)
    t_off = np.concatenate([[0], np.cumsum(ms)]).astype(np.int32)
    nt = int(t_off[-1])
    z = (rng.standard_normal((nt + B, V)) * 1.5).astype(np.float32)
    # scored columns: mostly inside the row's top 3, some anywhere
    cols = np.array([np.argsort(-z[i + b])[rng.integers(0, 3)] if rng.random() < 0.8
                     else rng.integers(0, V) for b in range(B)
                     for i in range(t_off[b], t_off[b + 1])], dtype=np.int32)
    qh = rng.uniform(0.05, 0.9, size=nt)
    out = oracle.verify(t_off, cols, qh, z, temp_target=T, seed=seed, top_k_target=k,
                        top_p_target=p)
    checked = rejected = 0
    for b in range(B):
        if out["boundary"][b]:
            continue
        t0, m, row0 = int(t_off[b]), int(ms[b]), int(t_off[b]) + b
        PF = [_kept_by_hand(z[row0 + j], T, k, p) for j in range(m + 1)]
        a = m
        for j in range(m):
            u = _np_uniform(seed, j, 0, b)
            if not u < PF[j][cols[t0 + j]] / qh[t0 + j]:
                a = j
                break
        assert out["accepted"][b] == a, b
        r = PF[a].copy()
        if a < m:
            t = cols[t0 + a]
            r[t] = max(0.0, r[t] - qh[t0 + a])
            rejected += 1
            if not r.sum() > 0:
                r = PF[a].copy()
        u2 = _np_uniform(seed, a, 1, b)
        x = int(np.argmax(np.cumsum(r) > u2 * r.sum()))
        assert r[x] > 0 and out["next_token"][b] == x, b
        assert np.allclose(out["p_hat"][t0:t0 + m], [PF[j][cols[t0 + j]] for j in range(m)],
                           atol=1e-12)
        checked += 1
    assert checked > 250 and rejected > 100
