"""Pins of the oracle's token distance and DTW (App. H, §4.1, Alg. 1) against
facts that do not come from the oracle itself: textbook values, the edit
distance's own definition searched by brute force, the worked example printed
in the paper, and exhaustive enumeration of warping paths."""
import itertools
import json
import os
import random
from collections import deque

import numpy as np
import pytest

import oracle

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


# ----------------------------------------------------------------- Levenshtein

@pytest.mark.parametrize("s,t,d", [
    (b"kitten", b"sitting", 3),  # the classic textbook pair
    (b"flaw", b"lawn", 2),
    (b"", b"", 0),
    (b"", b"abc", 3),
    (b"abc", b"", 3),
    (b"abc", b"abc", 0),
    (b"a", b"b", 1),
    (b"Saturday", b"Sunday", 3),
])
def test_lev_textbook_values(s, t, d):
    assert oracle.lev(s, t) == d


def _edit_distance_bfs(s: bytes, t: bytes, alphabet: bytes) -> int:
    """Minimum number of single-byte insertions, deletions and substitutions
    turning s into t, by breadth-first search over strings (App. H's definition
    of the distance, independent of its dynamic program)."""
    limit = len(s) + len(t)
    seen = {s: 0}
    q = deque([s])
    while q:
        u = q.popleft()
        du = seen[u]
        if u == t:
            return du
        if du >= limit:
            continue
        nxt = []
        for p in range(len(u) + 1):
            for c in alphabet:
                nxt.append(u[:p] + bytes([c]) + u[p:])
        for p in range(len(u)):
            nxt.append(u[:p] + u[p + 1:])
            for c in alphabet:
                nxt.append(u[:p] + bytes([c]) + u[p + 1:])
        for v in nxt:
            if len(v) <= max(len(s), len(t)) + 1 and v not in seen:
                seen[v] = du + 1
                q.append(v)
    raise AssertionError("unreachable")


def test_lev_matches_definition_by_search():
    rng = random.Random(5)
    alphabet = b"ab"
    for _ in range(60):
        s = bytes(rng.choice(alphabet) for _ in range(rng.randint(0, 4)))
        t = bytes(rng.choice(alphabet) for _ in range(rng.randint(0, 4)))
        assert oracle.lev(s, t) == _edit_distance_bfs(s, t, alphabet), (s, t)


def test_lev_metric_invariants():
    rng = random.Random(11)
    for _ in range(300):
        s, t, u = (bytes(rng.randrange(4) + 97 for _ in range(rng.randint(0, 9)))
                   for _ in range(3))
        dst = oracle.lev(s, t)
        assert oracle.lev(s, s) == 0
        assert dst == oracle.lev(t, s)
        assert abs(len(s) - len(t)) <= dst <= max(len(s), len(t))
        assert oracle.lev(s, u) <= dst + oracle.lev(t, u)
        assert oracle.lev(s, b"") == len(s)


def test_lev_is_byte_level_and_case_sensitive():
    assert oracle.lev("é".encode(), "e".encode()) == 2  # two UTF-8 bytes vs one
    assert oracle.lev(b"Law", b"law") == 1


# ------------------------------------------------------------------------ DTW

def _cost(a, b):
    return np.array([[oracle.lev(x.encode(), y.encode()) for y in b] for x in a], dtype=np.int32)


def test_fig2_worked_example():
    g = json.load(open(os.path.join(GOLDEN, "fig2_example.json")))
    D, T = g["draft_tokens"], g["target_tokens"]
    want = [(D.index(a), T.index(b)) for a, b in g["path_tokens"]]
    for w in (1, 2, 8, -1):
        cstar, path = oracle.dtw(_cost(D, T), w)
        assert path == want, w
        # C* is the sum of the local costs along the printed path (hand check:
        # d(S,Scale)=4, d(cal,Scale)=2, d(ing,ing)=0, d(Law,L)=2, d(Law,aw)=1)
        assert cstar == 9
    # transfer rule on the example: target j takes the last draft token aligned to it
    al = _align_strings(D, T, 8)
    assert list(al["map"]) == [1, 2, 3, 3]


def _align_strings(D, T, w):
    from paper_2510_15545_gb300.workload import Vocab
    vd = Vocab.from_strings([s.encode() for s in D])
    vt = Vocab.from_strings([s.encode() for s in T])
    return oracle.align([0, len(D)], list(range(len(D))), [0, len(T)], list(range(len(T))),
                        vd.blob, vd.off, vt.blob, vt.off, w)


def test_identical_sequences_give_diagonal_at_zero_cost():
    rng = np.random.default_rng(3)
    for n in (1, 2, 5, 17):
        toks = [bytes(rng.integers(97, 101, size=rng.integers(1, 6)).astype(np.uint8))
                for _ in range(n)]
        d = np.array([[oracle.lev(a, b) for b in toks] for a in toks], dtype=np.int32)
        for w in (0, 3, -1):
            cstar, path = oracle.dtw(d, w)
            assert cstar == 0
            assert path == [(i, i) for i in range(n)]


def _all_paths(k, m, band):
    """Every monotone warping path (1,1) -> (k,m) with unit steps inside |i-j| <= band,
    as a list of 1-based cells."""
    out = []

    def rec(i, j, acc):
        if (i, j) == (k, m):
            out.append(list(acc))
            return
        for di, dj in ((1, 1), (1, 0), (0, 1)):
            a, b = i + di, j + dj
            if a <= k and b <= m and abs(a - b) <= band:
                acc.append((a, b))
                rec(a, b, acc)
                acc.pop()

    rec(1, 1, [(1, 1)])
    return out


def _preferred_optimum(paths, d):
    """Among minimum-cost paths, the one whose predecessor choices read from the
    end are best under the order diagonal < up < left."""
    rank = {(1, 1): 0, (1, 0): 1, (0, 1): 2}

    def key(p):
        steps = [rank[(p[x][0] - p[x - 1][0], p[x][1] - p[x - 1][1])] for x in range(len(p) - 1, 0, -1)]
        return steps

    costs = [sum(int(d[i - 1, j - 1]) for i, j in p) for p in paths]
    best = min(costs)
    opt = [p for p, c in zip(paths, costs) if c == best]
    return best, min(opt, key=key)


@pytest.mark.parametrize("seed", range(40))
def test_dtw_against_path_enumeration(seed):
    rng = np.random.default_rng(seed)
    k, m = int(rng.integers(1, 7)), int(rng.integers(1, 7))
    d = rng.integers(0, 4, size=(k, m)).astype(np.int32)  # small range: many ties
    for w in (-1, 0, 1, 2):
        band = (k + m) if w < 0 else max(w, abs(k - m))
        best, pref = _preferred_optimum(_all_paths(k, m, band), d)
        cstar, path = oracle.dtw(d, w)
        assert cstar == best
        assert path == [(i - 1, j - 1) for i, j in pref]


def test_band_excludes_far_cells():
    # a zero-cost cell far off the diagonal is usable without a band only
    k = m = 6
    d = np.full((k, m), 5, dtype=np.int32)
    np.fill_diagonal(d, 1)
    d[0, 5] = d[5, 0] = 0
    c_band, p_band = oracle.dtw(d, 1)
    assert all(abs(i - j) <= 1 for i, j in p_band)
    assert c_band == 6
    c_free, _ = oracle.dtw(d, -1)
    assert c_free <= c_band


def test_unequal_lengths_widen_the_band():
    # |k - m| > w: the band grows to |k - m| so (k, m) stays reachable
    d = np.ones((2, 9), dtype=np.int32)
    cstar, path = oracle.dtw(d, 1)
    assert cstar == 9 and path[0] == (0, 0) and path[-1] == (1, 8)


def test_map_is_last_aligned_draft_index():
    # one-to-many: draft "ab" -> target "a","b" copies; many-to-one: "a","b" -> "ab"
    al = _align_strings(["ab", "c"], ["a", "b", "c"], 8)
    assert list(al["map"]) == [0, 0, 1]
    al = _align_strings(["a", "b", "c"], ["ab", "c"], 8)
    assert list(al["map"]) == [1, 2]


def test_align_status_codes():
    from paper_2510_15545_gb300.workload import Vocab
    v = Vocab.from_strings([b"a", b"b", b"x" * 300])
    out = oracle.align([0, 1, 1, 2, 3, 4, 5], [0, 0, 5, 0, 7], [0, 1, 2, 2, 3, 4, 5],
                       [1, 0, 1, 2, 2], v.blob, v.off, v.blob, v.off, 8)
    # 0 fine; 1 empty draft; 2 empty target; 3 id out of range; 4 token over 256
    # bytes; 5 both of the last two (every flag is reported)
    assert list(out["status"]) == [0, oracle.ST_EMPTY, oracle.ST_EMPTY, oracle.ST_ID_RANGE,
                                   oracle.ST_TOO_LONG, oracle.ST_ID_RANGE | oracle.ST_TOO_LONG]
    assert out["path_len"][0] == 1 and list(out["path_len"][1:]) == [0] * 5
