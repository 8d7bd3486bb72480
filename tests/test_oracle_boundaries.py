"""Pins of where the oracle says a boundary case lies, and of the comparison
that uses it (CPU only).

The parity contract excuses a device result that differs from the oracle's
only at the decision that lay within 1e-6 of its boundary (Alg. 4's accept
test u < min(1, p/q) and its inverse-CDF draw from the residual; the top-p cut
of the sampling filters, App. F). These tests recompute those locations by hand
from the definitions (numpy's Philox for the uniforms, scipy's softmax for the
rows) on inputs built to sit on a boundary, and plant mistakes in copies of
the oracle's outputs to show that the comparison excuses exactly the flagged
decision and nothing else."""
import numpy as np
from scipy import special

import oracle
from oracle.compare import compare_step

from test_oracle_sampling import _np_uniform


def _csr(ms):
    return np.concatenate([[0], np.cumsum(ms)]).astype(np.int32)


def test_accept_boundary_flag_sits_on_the_decision_it_concerns():
    """q_hat is set so that position jb's ratio p/q lies 5e-7 from its uniform;
    row_bnd bit 1 must be set on that row (if the decision was reached) and on
    no row whose |u - min(1, p/q)| is at least 1e-6."""
    rng = np.random.default_rng(5)
    B, V, seed = 200, 9, 4242
    ms = rng.integers(2, 7, size=B)
    t_off = _csr(ms)
    nt = int(t_off[-1])
    cols = rng.integers(0, V, size=nt).astype(np.int32)
    z = (rng.standard_normal((nt + B, V)) * 1.5).astype(np.float32)
    qh = np.zeros(nt)
    jb = np.zeros(B, int)
    for b in range(B):
        t0, m, row0 = int(t_off[b]), int(ms[b]), int(t_off[b]) + b
        P = special.softmax(z[row0:row0 + m].astype(np.float64), axis=1)
        jb[b] = rng.integers(0, m)
        for j in range(m):
            p = P[j, cols[t0 + j]]
            u = _np_uniform(seed, j, 0, b)
            if j < jb[b]:
                qh[t0 + j] = p * 0.5  # ratio 2: accepted, far from any boundary
            elif j == jb[b]:
                qh[t0 + j] = p / (u + (5e-7 if b % 2 else -5e-7))  # 5e-7 from u
            else:
                qh[t0 + j] = rng.uniform(0.05, 0.9)
    out = oracle.verify(t_off, cols, qh, z, seed=seed)
    hits = 0
    for b in range(B):
        t0, m, row0 = int(t_off[b]), int(ms[b]), int(t_off[b]) + b
        P = special.softmax(z[row0:row0 + m].astype(np.float64), axis=1)
        want = np.zeros(m + 1, bool)
        a = m
        for j in range(m):
            u = _np_uniform(seed, j, 0, b)
            acc = min(1.0, P[j, cols[t0 + j]] / qh[t0 + j])
            want[j] = abs(u - acc) < 1e-6
            if not u < acc:
                a = j
                break
        assert out["accepted"][b] == a
        got = (out["row_bnd"][row0:row0 + m + 1] & 1) != 0
        assert np.array_equal(got, want), (b, got, want)
        assert bool(out["boundary"][b] & 1) == bool(want.any())
        hits += bool(want[jb[b]])
    assert hits == B  # every planted decision was reached and flagged


def test_token_boundary_interval_is_the_columns_near_the_draw():
    """A bonus row whose first column's mass ends 3e-7 above the draw u' and
    whose second column is tiny: columns 0 and 1 are the boundary columns, the
    drawn token is 0; a row far from the draw reports no interval."""
    B, seed = 40, 99
    V = 4
    t_off = np.arange(B + 1, dtype=np.int32)  # m = 1 per request
    cols = np.zeros(B, np.int32)
    z = np.zeros((2 * B, V), np.float32)
    for b in range(B):
        u2 = _np_uniform(seed, 1, 1, b)  # all accepted: row a = 1 is drawn
        if b % 2 == 0:
            p0 = u2 + 3e-7
            p1 = 1e-9
        else:
            p0 = u2 * 0.5 + 0.25 * (1 - u2)  # far from the draw
            p1 = 0.1 * (1 - p0)
        rest = (1 - p0 - p1) / 2
        z[2 * b + 1] = np.log(np.array([p0, p1, rest, rest]))
        z[2 * b] = np.log(np.array([0.7, 0.1, 0.1, 0.1]))
    qh = np.full(B, 1e-3)  # p/q > 1: accepted
    out = oracle.verify(t_off, cols, qh, z, seed=seed)
    for b in range(B):
        assert out["accepted"][b] == 1
        r = special.softmax(z[2 * b + 1].astype(np.float64))
        theta = _np_uniform(seed, 1, 1, b) * r.sum()
        cum = np.cumsum(r)
        near = np.nonzero(np.abs(theta - cum) < 1e-6 * r.sum())[0]
        lo, hi = (int(near[0]), int(near[-1])) if len(near) else (-1, -1)
        assert (out["tok_lo"][b], out["tok_hi"][b]) == (lo, hi), b
        assert out["next_token"][b] == int(np.argmax(cum > theta))
        if b % 2 == 0:
            assert (lo, hi) == (0, 1)
        else:
            assert (lo, hi) == (-1, -1)


def test_filter_ambiguity_is_flagged_on_its_own_row():
    """A row with probabilities (0.5, 0.3, 0.2) cut at top-p 0.8 has the mass
    0.8 before its last token: ambiguous. Only that row carries bit 4, in
    verification (target rows) and in the transfer (draft rows)."""
    V = 3
    amb = np.log(np.array([0.5, 0.3, 0.2])).astype(np.float32)
    clear = np.log(np.array([0.6, 0.3, 0.1])).astype(np.float32)
    t_off = np.array([0, 2], np.int32)
    z = np.stack([clear, amb, clear])
    out = oracle.verify(t_off, np.array([0, 1], np.int32), np.array([0.9, 0.9]), z, seed=3,
                        top_k_target=3, top_p_target=0.8)
    assert list(out["row_bnd"] & 4) == [0, 4, 0]
    zd = np.stack([amb, clear, amb, clear])
    d_off = np.array([0, 4], np.int32)
    tr = oracle.transfer(d_off, np.zeros(4, np.int32), t_off, np.array([1, 2], np.int32), zd,
                         top_k=3, top_p=0.8)
    assert list(tr["drow_bnd"] & 4) == [0, 0, 4, 0]  # only mapped rows are evaluated


# ------------------------------------------------- the comparison, planted

def _case():
    """A small oracle step with enough requests to plant mistakes in copies."""
    rng = np.random.default_rng(8)
    B, V, seed = 60, 7, 515
    ms = rng.integers(2, 6, size=B)
    t_off = _csr(ms)
    nt = int(t_off[-1])
    cols = rng.integers(0, V, size=nt).astype(np.int32)
    z = (rng.standard_normal((nt + B, V)) * 1.5).astype(np.float32)
    qh = rng.uniform(0.05, 0.5, size=nt)
    o = oracle.verify(t_off, cols, qh, z, seed=seed)
    o["q_hat"] = qh
    d_off = t_off.copy()
    return o, d_off, t_off


def _cmp(g, o, d_off, t_off):
    return compare_step(g, o, d_off, t_off, check_align=False)


def _copy(o):
    return {k: np.array(v, copy=True) for k, v in o.items()}


def test_comparison_accepts_the_oracle_itself():
    o, d_off, t_off = _case()
    r = _cmp(_copy(o), o, d_off, t_off)
    assert r["mismatches"] == [] and r["accept_boundary"] == 0 and r["token_boundary"] == 0


def test_comparison_excuses_an_accept_difference_only_at_the_flagged_decision():
    o, d_off, t_off = _case()
    b = int(np.nonzero(o["accepted"] >= 2)[0][0])
    row0 = int(t_off[b]) + b
    a = int(o["accepted"][b])
    g = _copy(o)
    g["accepted"][b] = a - 1  # disagree first at decision a - 1
    assert len(_cmp(g, o, d_off, t_off)["mismatches"]) == 1  # nothing flagged: caught
    o2 = _copy(o)
    o2["row_bnd"][row0 + a - 2] |= 1  # a flag on another decision does not excuse it
    assert len(_cmp(g, o2, d_off, t_off)["mismatches"]) == 1
    o2["row_bnd"][row0 + a - 1] |= 1  # the flag on the decision that differs does
    r = _cmp(g, o2, d_off, t_off)
    assert r["mismatches"] == [] and r["accept_boundary"] == 1


def test_comparison_excuses_a_token_difference_only_inside_the_boundary_columns():
    o, d_off, t_off = _case()
    b = 3
    t = int(o["next_token"][b])
    g = _copy(o)
    g["next_token"][b] = t + 1 if t < 6 else t - 1
    assert len(_cmp(g, o, d_off, t_off)["mismatches"]) == 1
    o2 = _copy(o)
    o2["tok_lo"][b] = o2["tok_hi"][b] = min(t, int(g["next_token"][b]))
    r = _cmp(g, o2, d_off, t_off)
    assert r["mismatches"] == [] and r["token_boundary"] == 1
    g["next_token"][b] = (t + 3) % 7  # two columns away: outside the interval
    assert len(_cmp(g, o2, d_off, t_off)["mismatches"]) == 1


def test_comparison_bounds_small_probabilities_relatively():
    o, d_off, t_off = _case()
    g = _copy(o)
    o2 = _copy(o)
    o2["p_hat"][0] = 1e-8
    g["p_hat"][0] = 2e-8  # within 1e-5 absolute, 100% off: caught
    assert len(_cmp(g, o2, d_off, t_off)["mismatches"]) == 1
    g["p_hat"][0] = 1e-8 * (1 + 5e-5)  # within both bounds
    assert _cmp(g, o2, d_off, t_off)["mismatches"] == []
    g = _copy(o)
    g["lse"][5] += 2e-5  # lse is bounded absolutely
    assert len(_cmp(g, o, d_off, t_off)["mismatches"]) == 1


def test_comparison_excuses_filter_ambiguity_only_on_its_row():
    o, d_off, t_off = _case()
    b = int(np.nonzero(o["accepted"] >= 1)[0][0])
    row0 = int(t_off[b]) + b
    g = _copy(o)
    g["p_hat"][t_off[b] + 1] += 0.01
    assert len(_cmp(g, o, d_off, t_off)["mismatches"]) == 1
    o2 = _copy(o)
    o2["row_bnd"][row0] |= 4  # row 0 ambiguous does not excuse row 1
    assert len(_cmp(g, o2, d_off, t_off)["mismatches"]) == 1
    o2["row_bnd"][row0 + 1] |= 4
    assert _cmp(g, o2, d_off, t_off)["mismatches"] == []
