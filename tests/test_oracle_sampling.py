"""Pins of the oracle's random numbers, softmax, transfer and verification
against independent libraries (numpy's Philox, scipy's softmax) and against
what speculative sampling guarantees mathematically (Alg. 4: the emitted token
is distributed as p; accepted lengths follow the product of min(1, p/q))."""
import numpy as np
import pytest
import torch
from scipy import special, stats

import oracle

MASK64 = (1 << 64) - 1


# --------------------------------------------------------------------- Philox

def test_philox_known_answer():
    # Random123's published known-answer vector for philox4x64-10, zero counter and key
    assert oracle.philox4x64_10([0, 0, 0, 0], [0, 0]) == [
        0x16554D9ECA36314C, 0xDB20FE9D672D0FDC, 0xD7E772CEE186176B, 0x7E68B68AEC7BA23B]


@pytest.mark.parametrize("ctr,key", [
    ([1, 0, 0, 0], [1234, 0]),
    ([7, 1, 63, 0], [1234, 0]),
    ([0, 0, 5, 0], [99, 0]),
    ([0, 1, 0, 0], [2**63 + 5, 17]),
    ([123456789, 1, 2**40 + 3, 0], [0xDEADBEEF, 0]),
])
def test_philox_matches_numpy(ctr, key):
    # numpy's Philox is Philox4x64-10 and advances the 256-bit counter by one
    # before producing a block, so it is seeded with counter - 1.
    c = sum(v << (64 * i) for i, v in enumerate(ctr)) - 1
    c &= (1 << 256) - 1
    words = np.array([(c >> (64 * i)) & MASK64 for i in range(4)], dtype=np.uint64)
    g = np.random.Philox(key=np.array(key, dtype=np.uint64), counter=words)
    want = [int(x) for x in g.random_raw(4)]
    assert oracle.philox4x64_10(ctr, key) == want


def test_uniform_is_top_24_bits():
    for pos, stream, req in [(0, 0, 0), (3, 1, 9), (511, 0, 4095)]:
        w = oracle.philox4x64_10([pos, stream, req, 0], [1234, 0])[0]
        u = oracle.uniform(1234, pos, stream, req)
        assert u == (w >> 40) / 2.0**24
        assert 0.0 <= u < 1.0


def test_uniforms_are_uniform():
    us = np.array([oracle.uniform(7, j, s, b) for j in range(20) for s in (0, 1)
                   for b in range(250)])
    assert stats.kstest(us, "uniform").pvalue > 1e-3


# -------------------------------------------------------------------- softmax

@pytest.mark.parametrize("T", [1.0, 0.6, 1.7])
def test_softmax_and_lse_against_scipy(T):
    rng = np.random.default_rng(0)
    # on a 2^-10 grid, so that the shift below is exact in fp32
    z = (np.round(rng.standard_normal(5000) * 4 * 1024) / 1024).astype(np.float32)
    p = oracle.softmax(z, T)
    want = special.softmax(z.astype(np.float64) / T)
    assert np.max(np.abs(p - want)) < 1e-15
    assert abs(p.sum() - 1) < 1e-12
    assert abs(oracle.logsumexp(z, T) - special.logsumexp(z.astype(np.float64) / T)) < 1e-12
    # shift invariance
    p2 = oracle.softmax(z + np.float32(8.0), T)
    assert np.max(np.abs(p2 - p)) < 1e-12


def test_bf16_rows_are_decoded_exactly():
    z = torch.tensor([1.0, -2.0, 0.5, 3.140625], dtype=torch.bfloat16)
    want = special.softmax(np.array([1.0, -2.0, 0.5, 3.140625]))
    assert np.max(np.abs(oracle.softmax(z) - want)) < 1e-15


# ------------------------------------------------------------------- transfer

def test_transfer_is_softmax_at_mapped_draft_token():
    rng = np.random.default_rng(1)
    V, k = 300, 5
    logits = (rng.standard_normal((k, V)) * 2).astype(np.float32)
    cols = rng.integers(0, V, size=k).astype(np.int32)
    mp = np.array([0, 0, 2, 3, 4, 4], dtype=np.int32)  # one-to-many copies and a skip
    out = oracle.transfer([0, k], cols, [0, len(mp)], mp, logits, 0.8)
    for j, i in enumerate(mp):
        assert abs(out["q_hat"][j] - special.softmax(logits[i].astype(np.float64) / 0.8)[cols[i]]) < 1e-15
    probs = rng.random(k).astype(np.float32)
    out = oracle.transfer([0, k], cols, [0, len(mp)], mp, None, 1.0, draft_probs=probs)
    assert np.array_equal(out["q_hat"], probs[mp].astype(np.float64))


# --------------------------------------------------------------- verification

def _rows(p):
    """Logit rows whose softmax is exactly the given probability rows (up to
    fp32 rounding of the log)."""
    return np.log(np.asarray(p, dtype=np.float64)).astype(np.float32)


def test_full_q_emits_the_target_distribution():
    """Alg. 4 losslessness: draft t ~ q, accept with min(1, p/q), else resample
    from the normalised max(0, p - q): the emitted token is distributed as p."""
    rng = np.random.default_rng(2)
    V, N = 12, 40000
    p = rng.dirichlet(np.ones(V) * 0.7)
    q = rng.dirichlet(np.ones(V) * 0.7)
    zp, zq = _rows(p), _rows(q)
    p32, q32 = special.softmax(zp.astype(np.float64)), special.softmax(zq.astype(np.float64))
    t = rng.choice(V, size=N, p=q32)
    target_off = np.arange(N + 1, dtype=np.int32)
    tl = np.empty((2 * N, V), dtype=np.float32)
    tl[0::2] = zp
    tl[1::2] = zp  # bonus rows (not used for the first emitted token)
    dl = np.broadcast_to(zq, (N, V)).copy()
    q_hat = q32[t]
    out = oracle.verify(target_off, t.astype(np.int32), q_hat, tl, seed=77, full_q=True,
                        draft_off=target_off, mp=np.zeros(N, np.int32), draft_logits=dl)
    first = np.where(out["accepted"] == 1, t, out["next_token"])
    counts = np.bincount(first, minlength=V)
    assert stats.chisquare(counts, p32 * N).pvalue > 1e-4
    # the draft distribution itself is far from p, so the test has power
    assert stats.chisquare(np.bincount(t, minlength=V), p32 * N).pvalue < 1e-6


def test_one_hot_residual_closed_form():
    """One-hot transfer: with drafted token t and q_hat > p(t), the first emitted
    token is t with probability p(t)/q_hat, otherwise x != t with probability
    proportional to p(x) (the residual max(0, p - q_hat e_t))."""
    rng = np.random.default_rng(3)
    V, N, t = 10, 40000, 4
    p = rng.dirichlet(np.ones(V))
    zp = _rows(p)
    p32 = special.softmax(zp.astype(np.float64))
    qh = min(1.0, p32[t] * 2.5)
    tl = np.repeat(zp[None, :], 2 * N, axis=0)
    out = oracle.verify(np.arange(N + 1, dtype=np.int32), np.full(N, t, np.int32),
                        np.full(N, qh), tl, seed=5)
    first = np.where(out["accepted"] == 1, t, out["next_token"])
    acc = p32[t] / qh
    want = (1 - acc) * p32 / (1 - p32[t])
    want[t] = acc
    assert stats.chisquare(np.bincount(first, minlength=V), want * N).pvalue > 1e-4


def test_accepted_length_distribution():
    """P(a >= j) is the product of min(1, p_l / q_l) over l <= j."""
    rng = np.random.default_rng(4)
    V, m, N = 16, 4, 20000
    zs = (rng.standard_normal((m + 1, V)) * 1.5).astype(np.float32)
    cols = rng.integers(0, V, size=m).astype(np.int32)
    ph = np.array([special.softmax(zs[j].astype(np.float64))[cols[j]] for j in range(m)])
    qh = ph / np.array([0.9, 0.5, 1.3, 0.7])  # acceptance probabilities .9 .5 1 .7
    tl = np.tile(zs, (N, 1))
    out = oracle.verify(np.arange(0, m * N + 1, m, dtype=np.int32), np.tile(cols, N),
                        np.tile(qh, N), tl, seed=11)
    a = out["accepted"]
    surv = np.cumprod(np.minimum(1, ph / qh))
    for j in range(1, m + 1):
        emp = np.mean(a >= j)
        sd = np.sqrt(surv[j - 1] * (1 - surv[j - 1]) / N) + 1e-12
        assert abs(emp - surv[j - 1]) < 5 * sd, (j, emp, surv[j - 1])
    assert np.allclose(out["p_hat"][:m], ph, atol=1e-15)
    assert np.allclose(out["lse"][:m + 1], special.logsumexp(zs.astype(np.float64), axis=1))


def test_bonus_row_when_all_accepted():
    # q_hat tiny: every draft is accepted and the next token comes from row m
    V, N = 6, 30000
    p = np.array([0.05, 0.4, 0.1, 0.2, 0.15, 0.1])
    zp = _rows(p)
    bonus = _rows(np.array([0.5, 0.1, 0.1, 0.1, 0.1, 0.1]))
    tl = np.empty((2 * N, V), np.float32)
    tl[0::2] = zp
    tl[1::2] = bonus
    out = oracle.verify(np.arange(N + 1, dtype=np.int32), np.ones(N, np.int32),
                        np.full(N, 1e-9), tl, seed=3)
    assert np.all(out["accepted"] == 1)
    want = special.softmax(bonus.astype(np.float64)) * N
    assert stats.chisquare(np.bincount(out["next_token"], minlength=V), want).pvalue > 1e-4


def _np_uniform(seed, pos, stream, req):
    """u from numpy's own Philox4x64-10 at counter (pos, stream, req, 0), key
    (seed, 0): the top 24 bits of the block's first word times 2^-24."""
    c = (pos + (stream << 64) + (req << 128) - 1) & ((1 << 256) - 1)
    words = np.array([(c >> (64 * i)) & MASK64 for i in range(4)], dtype=np.uint64)
    g = np.random.Philox(key=np.array([seed, 0], dtype=np.uint64), counter=words)
    return (int(g.random_raw(1)[0]) >> 40) / 2.0**24


def test_each_decision_uses_its_own_uniform_and_the_inverse_cdf():
    """Every accept decision and every next token recomputed by hand from the
    definitions: u_j from numpy's Philox at (j, stream 0, request_base + b),
    accept while u_j < p_j / q_j, then the residual (p with t_a's mass lowered
    by q_hat, or the bonus row) sampled at u' from (a, stream 1, ...) as the
    smallest column whose running mass exceeds u' Z."""
    rng = np.random.default_rng(21)
    B, V, seed, base = 300, 12, 77, 1000
    ms = rng.integers(1, 6, size=B)
    t_off = np.concatenate([[0], np.cumsum(ms)]).astype(np.int32)
    nt = int(t_off[-1])
    cols = rng.integers(0, V, size=nt).astype(np.int32)
    z = (rng.standard_normal((nt + B, V)) * 1.2).astype(np.float32)
    qh = rng.uniform(0.02, 0.6, size=nt)
    out = oracle.verify(t_off, cols, qh, z, seed=seed, request_base=base)
    n_acc = n_rej = 0
    for b in range(B):
        if out["boundary"][b]:
            continue
        t0, m, row0 = int(t_off[b]), int(ms[b]), int(t_off[b]) + b
        P = special.softmax(z[row0:row0 + m + 1].astype(np.float64), axis=1)
        a = m
        for j in range(m):
            u = _np_uniform(seed, j, 0, base + b)
            if not u < P[j, cols[t0 + j]] / qh[t0 + j]:
                a = j
                break
        assert out["accepted"][b] == a, b
        r = P[a].copy()
        if a < m:
            t = cols[t0 + a]
            r[t] = max(0.0, r[t] - qh[t0 + a])
            n_rej += 1
        else:
            n_acc += 1
        u2 = _np_uniform(seed, a, 1, base + b)
        x = int(np.argmax(np.cumsum(r) > u2 * r.sum()))
        assert out["next_token"][b] == x, b
    assert n_acc > 20 and n_rej > 100  # both branches are exercised


def test_full_q_decisions_recomputed_by_hand():
    """Full-q mode (one vocabulary, Alg. 4 as printed): each rejection's next
    token comes from max(0, p_a - q) against the whole mapped draft row at T_d
    (the row itself when that has no mass), each bonus token from row m."""
    rng = np.random.default_rng(22)
    B, V, k, seed, Td, Tt = 250, 10, 4, 31, 0.8, 1.1
    ms = rng.integers(1, 6, size=B)
    t_off = np.concatenate([[0], np.cumsum(ms)]).astype(np.int32)
    d_off = np.arange(0, B * k + 1, k, dtype=np.int32)
    nt = int(t_off[-1])
    zt = (rng.standard_normal((nt + B, V)) * 1.3).astype(np.float32)
    zd = (rng.standard_normal((B * k, V)) * 1.3).astype(np.float32)
    mp = np.concatenate([np.sort(rng.integers(0, k, size=m)) for m in ms]).astype(np.int32)
    cols = rng.integers(0, V, size=nt).astype(np.int32)
    Q = special.softmax(zd.astype(np.float64) / Td, axis=1)
    qh = np.array([Q[d_off[b] + mp[j], cols[j]] for b in range(B)
                   for j in range(t_off[b], t_off[b + 1])])
    out = oracle.verify(t_off, cols, qh, zt, temp_target=Tt, seed=seed, full_q=True,
                        draft_off=d_off, mp=mp, draft_logits=zd, temp_draft=Td)
    rejected = 0
    for b in range(B):
        if out["boundary"][b]:
            continue
        t0, m, row0 = int(t_off[b]), int(ms[b]), int(t_off[b]) + b
        P = special.softmax(zt[row0:row0 + m + 1].astype(np.float64) / Tt, axis=1)
        a = m
        for j in range(m):
            if not _np_uniform(seed, j, 0, b) < P[j, cols[t0 + j]] / qh[t0 + j]:
                a = j
                break
        assert out["accepted"][b] == a, b
        r = P[a].copy()
        if a < m:
            r = np.maximum(0.0, P[a] - Q[d_off[b] + mp[t0 + a]])
            if not r.sum() > 0:
                r = P[a].copy()
            rejected += 1
        u2 = _np_uniform(seed, a, 1, b)
        assert out["next_token"][b] == int(np.argmax(np.cumsum(r) > u2 * r.sum())), b
    assert rejected > 100


def test_rejected_token_is_never_resampled():
    V, N = 5, 2000
    zp = _rows([0.3, 0.2, 0.2, 0.2, 0.1])
    tl = np.repeat(zp[None, :], 2 * N, axis=0)
    out = oracle.verify(np.arange(N + 1, dtype=np.int32), np.zeros(N, np.int32),
                        np.full(N, 0.99), tl, seed=9)
    rej = out["accepted"] == 0
    assert rej.sum() > 1000
    assert np.all(out["next_token"][rej] != 0)


def test_verify_status_and_seed_dependence():
    V = 8
    tl = np.zeros((6, V), np.float32)
    out = oracle.verify([0, 2, 2, 3], [1, 9, 0], [0.5, 0.5, 0.5], tl)
    assert out["status"][0] == oracle.ST_ID_RANGE and out["next_token"][0] == -1
    assert out["status"][1] == oracle.ST_EMPTY
    assert out["status"][2] == 0 and 0 <= out["next_token"][2] < V
    N = 64
    tl = np.tile(_rows(np.full(V, 1 / V)), (2 * N, 1))
    args = (np.arange(N + 1, dtype=np.int32), np.zeros(N, np.int32), np.full(N, 0.5), tl)
    a = oracle.verify(*args, seed=1)
    b = oracle.verify(*args, seed=1)
    c = oracle.verify(*args, seed=2)
    assert np.array_equal(a["next_token"], b["next_token"])
    assert not np.array_equal(a["next_token"], c["next_token"])
    d = oracle.verify(*args, seed=1, request_base=N)
    assert not np.array_equal(a["next_token"], d["next_token"])
