"""Pins of the oracle's repetition penalty (the generation hyperparameter table,
App. F: the Qwen2.5-0.5B row sets a penalty of 1.1; the paper keeps each
model's Hugging Face defaults, whose rule is the one pinned here). A row's
penalized set is the request's history plus the sequence tokens before the
row's position; each of its columns has its logit z replaced by z * theta
when z < 0 and by z / theta otherwise, once, in fp32, before temperature and
the filters. CPU only."""
import numpy as np
import pytest

import oracle


def _verify(zt, cols, q, hist, theta, **kw):
    """One request: target rows zt (m + 1 rows), its m scored columns."""
    m = len(cols)
    return oracle.verify(np.array([0, m], np.int32), np.asarray(cols, np.int32),
                         np.asarray(q, np.float64), np.asarray(zt, np.float32),
                         rep_penalty_target=theta, hist_off_t=np.array([0, len(hist)], np.int32),
                         hist_cols_t=np.asarray(hist, np.int32), **kw)


def test_hand_worked_row():
    """z = (2, -1, 0.5, 1), history {0, 1}, theta = 2: the penalized row is
    (2 / 2, -1 * 2, 0.5, 1) = (1, -2, 0.5, 1). With e^1 = 2.718281828,
    e^-2 = 0.135335283, e^0.5 = 1.648721271 the normaliser is 7.220620211 and
    the probabilities are 0.376460990, 0.018742894, 0.228335131, 0.376460990
    (T = 1); at T = 0.5 the row is (2, -4, 1, 2) and they are 0.421877174,
    0.001045731, 0.155199942, 0.421877174."""
    row = [2.0, -1.0, 0.5, 1.0]
    for T, want in ((1.0, [0.376460990, 0.018742894, 0.228335131, 0.376460990]),
                    (0.5, [0.421877174, 0.001045731, 0.155199942, 0.421877174])):
        for c in range(4):
            out = _verify([row, row], [c], [0.5], [0, 1], 2.0, temp_target=T)
            assert abs(out["p_hat"][0] - want[c]) < 1e-8, (T, c, out["p_hat"][0])
        lse = np.log(np.exp(np.array([1.0, -2.0, 0.5, 1.0]) / T).sum())
        assert abs(out["lse"][0] - lse) < 1e-12


def test_no_penalty_and_empty_history_change_nothing():
    rng = np.random.default_rng(1)
    zt = rng.standard_normal((4, 50)).astype(np.float32) * 2
    cols = [3, 17, 3]
    base = _verify(zt, cols, [0.3, 0.2, 0.4], [], 1.0)
    same = _verify(zt, cols, [0.3, 0.2, 0.4], [5, 9], 1.0)
    assert np.array_equal(base["p_hat"], same["p_hat"])
    # a penalty with an empty history still penalizes the earlier sequence tokens
    pen = _verify(zt, cols, [0.3, 0.2, 0.4], [], 1.5)
    assert pen["p_hat"][0] == base["p_hat"][0]      # row 0: nothing before t_1
    assert pen["p_hat"][2] != base["p_hat"][2]      # row 2: t_3 = t_1 = column 3


def test_sign_rule_lowers_both_signs():
    """A positive logit is divided, a negative one multiplied: either way the
    penalized token loses probability (theta > 1), and with the rule reversed
    (dividing a negative logit) it would gain it."""
    for z0 in (1.5, -1.5):
        row = np.array([z0, 0.2, -0.3, 0.1], np.float32)
        plain = _verify([row, row], [0], [0.5], [], 1.0)["p_hat"][0]
        pen = _verify([row, row], [0], [0.5], [0], 1.3)["p_hat"][0]
        z1 = np.float32(z0) * np.float32(1.3) if z0 < 0 else np.float32(z0) / np.float32(1.3)
        e = np.exp(np.array([z1, 0.2, -0.3, 0.1], np.float32).astype(np.float64))
        assert pen < plain
        assert abs(pen - e[0] / e.sum()) < 1e-12


def test_each_column_once_however_often_it_occurs():
    rng = np.random.default_rng(2)
    zt = rng.standard_normal((3, 40)).astype(np.float32) * 3
    once = _verify(zt, [4, 8], [0.4, 0.4], [7, 11], 1.2)
    many = _verify(zt, [4, 8], [0.4, 0.4], [7, 11, 7, 7, 11], 1.2)
    assert np.array_equal(once["p_hat"], many["p_hat"])
    assert np.array_equal(once["lse"], many["lse"])
    # a history column that is also an earlier sequence token: penalized once
    both = _verify(zt, [4, 4], [0.4, 0.4], [4], 1.2)
    z = zt[1].copy()
    z[4] = z[4] * np.float32(1.2) if z[4] < 0 else z[4] / np.float32(1.2)
    e = np.exp(z.astype(np.float64))
    assert abs(both["p_hat"][1] - e[4] / e.sum()) < 1e-15


def test_the_penalized_set_grows_along_the_sequence():
    """Target row j scores t_{j+1}; t_1..t_j join the history for it, t_{j+1}
    itself does not."""
    V = 30
    rng = np.random.default_rng(3)
    row = (rng.standard_normal(V) * 2).astype(np.float32)
    row[12] = 4.0
    zt = np.stack([row] * 4)
    out = _verify(zt, [12, 12, 3], [0.2, 0.2, 0.2], [], 1.25)
    e = np.exp(row.astype(np.float64))
    assert abs(out["p_hat"][0] - e[12] / e.sum()) < 1e-12   # row 0: nothing penalized
    pen = row.copy()
    pen[12] = np.float32(4.0) / np.float32(1.25)
    e2 = np.exp(pen.astype(np.float64))
    assert abs(out["p_hat"][1] - e2[12] / e2.sum()) < 1e-12  # row 1: t_1 = 12 penalized
    pen3 = pen.copy()                                        # row 2: t_1, t_2 = {12}
    assert abs(out["p_hat"][2] - np.exp(pen3[3].astype(np.float64)) /
               np.exp(pen3.astype(np.float64)).sum()) < 1e-12


def test_penalized_logit_is_rounded_to_fp32():
    """1 / 1.1 is 0.9090909090909091 in fp64 and 0.90909094 in fp32: the
    penalized logit is the fp32 quotient of the fp32 operands."""
    row = np.array([1.0, 0.0, 0.0], np.float32)
    out = _verify([row, row], [0], [0.5], [0], 1.1)
    z = float(np.float32(1.0) / np.float32(1.1))
    assert z != 1.0 / 1.1
    want = np.exp(z) / (np.exp(z) + 2.0)
    assert abs(out["p_hat"][0] - want) < 1e-15
    bad = np.exp(1.0 / 1.1) / (np.exp(1.0 / 1.1) + 2.0)
    assert abs(out["p_hat"][0] - bad) > 1e-9


def test_draft_rows_penalize_the_draft_tokens_before_them():
    """The transfer's draft row i penalizes the history and d_1..d_i (draft
    columns of positions 0..i-1), never d_{i+1} itself."""
    V = 20
    rng = np.random.default_rng(4)
    zd = (rng.standard_normal((3, V)) * 2).astype(np.float32)
    d_cols = np.array([5, 5, 9], np.int32)
    mp = np.array([0, 1, 2], np.int32)
    out = oracle.transfer(np.array([0, 3], np.int32), d_cols, np.array([0, 3], np.int32), mp, zd,
                          1.0, rep_penalty=1.5, hist_off=np.array([0, 1], np.int32),
                          hist_cols=np.array([9], np.int32))
    def p(row, penal, c):
        z = row.copy()
        for x in penal:
            z[x] = z[x] * np.float32(1.5) if z[x] < 0 else z[x] / np.float32(1.5)
        e = np.exp(z.astype(np.float64))
        return e[c] / e.sum()
    assert abs(out["q_hat"][0] - p(zd[0], [9], 5)) < 1e-12
    assert abs(out["q_hat"][1] - p(zd[1], [9, 5], 5)) < 1e-12
    assert abs(out["q_hat"][2] - p(zd[2], [9, 5], 9)) < 1e-12


def test_history_statuses():
    zt = np.zeros((2, 10), np.float32)
    bad_col = _verify(zt, [1], [0.5], [10], 1.1)
    assert bad_col["status"][0] == oracle.ST_ID_RANGE
    out = oracle.verify(np.array([0, 1], np.int32), np.array([1], np.int32), np.array([0.5]),
                        zt, rep_penalty_target=1.1, hist_off_t=np.array([3, 1], np.int32),
                        hist_cols_t=np.array([0, 1, 2], np.int32))
    assert out["status"][0] == oracle.ST_BAD_OFFSETS


def test_filters_act_on_the_penalized_row():
    """Top-k after the penalty: a history token that leads the raw row drops
    out of the top 2 once penalized."""
    row = np.array([3.0, 2.9, 2.8, -1.0], np.float32)
    raw = _verify([row, row], [0], [0.5], [], 1.0, top_k_target=2)
    pen = _verify([row, row], [0], [0.5], [0], 1.2, top_k_target=2)
    assert raw["p_hat"][0] > 0.5
    assert pen["p_hat"][0] == 0.0  # 3.0 / 1.2 = 2.5 ranks third
