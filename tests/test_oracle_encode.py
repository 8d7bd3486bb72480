"""Pins of the oracle's re-encoding, Lemma-1 check and delta-pos histogram.

Re-encoding (section 4.2, App. A.1): T = encode_t(decode_d(D)) with greedy
longest match over the target vocabulary's byte strings. Pins: the paper's
'Scaling' example (section 2), brute-force maximality and Lemma 1 on random
vocabularies, agreement with the workload generator's own greedy encoder on the
synthetic vocabularies, and the status rules. Delta-pos (section 4.1, App. K):
hand-counted histograms of the Fig. 2 path.
"""
import json
import os

import numpy as np
import pytest

import oracle
from paper_2510_15545_gb300 import workload as W

HERE = os.path.dirname(os.path.abspath(__file__))


def table(strings):
    blob = b"".join(strings)
    off = np.zeros(len(strings) + 1, np.int64)
    off[1:] = np.cumsum([len(s) for s in strings])
    return np.frombuffer(blob, np.uint8).copy(), off


def concat(strings, ids):
    return b"".join(strings[i] for i in ids)


def test_scaling_example_from_the_paper():
    g = json.load(open(os.path.join(HERE, "golden", "scaling_example.json")))
    vd = [s.encode() for s in g["draft_vocab"]]
    vt = [bytes([i]) for i in range(256)] + [s.encode() for s in g["target_vocab_extra"]]
    D = [vd.index(s.encode()) for s in g["draft"]]
    r = oracle.encode([0, len(D)], D, *table(vd), *table(vt), max_m=16)
    assert r["status"].tolist() == [0]
    assert [vt[i].decode() for i in r["target_ids"]] == g["target"]


def random_vocab(rng, n, alphabet=b"abcde", max_len=6, all_bytes=True):
    out = [bytes([i]) for i in range(256)] if all_bytes else []
    seen = set(out)
    while len(out) < n:
        L = int(rng.integers(1, max_len + 1))
        s = bytes(rng.choice(list(alphabet), L).tolist())
        if s not in seen:
            seen.add(s)
            out.append(s)
    return out


def test_greedy_is_longest_match_and_lemma1():
    """At every emitted position no longer target token spells the next bytes
    (brute force over the whole vocabulary), and the bytes of T are those of D."""
    rng = np.random.default_rng(1)
    vd = random_vocab(rng, 300)
    vt = random_vocab(rng, 400)
    vt_set = {s: i for i, s in reversed(list(enumerate(vt)))}
    B = 40
    k = rng.integers(1, 12, B)
    off = np.concatenate([[0], np.cumsum(k)]).astype(np.int32)
    D = rng.integers(0, len(vd), int(off[-1])).astype(np.int32)
    r = oracle.encode(off, D, *table(vd), *table(vt), max_m=128)
    assert (r["status"] == 0).all()
    for b in range(B):
        text = concat(vd, D[off[b]:off[b + 1]])
        T = r["target_ids"][r["target_off"][b]:r["target_off"][b + 1]]
        assert concat(vt, T) == text  # Lemma 1
        p = 0
        for t in T:
            L = len(vt[t])
            assert vt_set[vt[t]] == t  # smallest id of its string
            for L2 in range(L + 1, len(text) - p + 1):
                assert text[p:p + L2] not in vt_set
            p += L


def test_smallest_id_among_equal_strings():
    vd = [b"ab"]
    vt = [b"x", b"ab", b"a", b"ab", b"b"]
    r = oracle.encode([0, 1], [0], *table(vd), *table(vt), max_m=4)
    assert r["target_ids"].tolist() == [1]


def test_no_match_and_limits():
    vd = [b"abc", b"z"]
    vt = [b"a", b"b", b"c", b"bc"]
    tv = table(vt)
    r = oracle.encode([0, 1, 2, 2], [0, 1], *table(vd), *tv, max_m=4)
    assert r["status"].tolist() == [0, oracle.ST_NO_MATCH, oracle.ST_EMPTY]
    assert r["target_ids"].tolist() == [0, 3]
    assert r["target_off"].tolist() == [0, 2, 2, 2]
    # more than max_m tokens
    r = oracle.encode([0, 1], [0], *table(vd), *tv, max_m=1)
    assert r["status"].tolist() == [oracle.ST_TOO_LONG]
    # decoded string longer than max_bytes
    r = oracle.encode([0, 1], [0], *table(vd), *tv, max_m=4, max_bytes=2)
    assert r["status"].tolist() == [oracle.ST_TOO_LONG]
    # id out of range, bad offsets
    r = oracle.encode([0, 1, 0], [5], *table(vd), *tv, max_m=4)
    assert r["status"].tolist() == [oracle.ST_ID_RANGE, oracle.ST_BAD_OFFSETS]


def test_capacity_counts_every_earlier_request():
    vd = [b"abc"]
    vt = [b"a", b"b", b"c"]
    off = [0, 1, 2, 3]
    r = oracle.encode(off, [0, 0, 0], *table(vd), *table(vt), max_m=4, capacity=7)
    # 3 + 3 fit, the third would end at 9 > 7
    assert r["status"].tolist() == [0, 0, oracle.ST_TOO_LONG]
    assert r["target_off"].tolist() == [0, 3, 6, 6]


@pytest.mark.parametrize("name", ["b1_g4_v32k", "b64_g8_v152k"])
def test_matches_the_generators_greedy_encoder(name):
    """Another implementation of the same rule (the workload generator's, used
    to build vocabularies and check coverage) gives the same tokens."""
    wl = W.make_workload(name, B=8, seed=3)
    r = oracle.encode(wl.draft_off, wl.draft_ids, wl.vd.blob, wl.vd.off, wl.vt.blob, wl.vt.off,
                      max_m=512)
    assert (r["status"] == 0).all()
    for b in range(wl.B):
        text = b"".join(wl.vd.strings[i] for i in wl.draft_ids[wl.draft_off[b]:wl.draft_off[b + 1]])
        want = W.greedy_encode(text, wl.vt.index)
        got = r["target_ids"][r["target_off"][b]:r["target_off"][b + 1]].tolist()
        assert got == want


def test_consistency_check():
    vd = [b"Scal", b"ing"]
    vt = [b"Scaling", b"Scal", b"ing", b"S", b"x"]
    tvd, tvt = table(vd), table(vt)
    ok = oracle.consistency([0, 2], [0, 1], [0, 1], [0], *tvd, *tvt, 8, 8)
    assert ok.tolist() == [0]
    ok = oracle.consistency([0, 2], [0, 1], [0, 2], [1, 2], *tvd, *tvt, 8, 8)
    assert ok.tolist() == [0]
    bad = oracle.consistency([0, 2], [0, 1], [0, 2], [1, 4], *tvd, *tvt, 8, 8)
    assert bad.tolist() == [oracle.ST_INCONSISTENT]
    short = oracle.consistency([0, 2], [0, 1], [0, 1], [3], *tvd, *tvt, 8, 8)
    assert short.tolist() == [oracle.ST_INCONSISTENT]
    longer = oracle.consistency([0, 1], [0], [0, 1], [0], *tvd, *tvt, 8, 8)
    assert longer.tolist() == [oracle.ST_INCONSISTENT]
    assert oracle.consistency([0, 2], [0, 1], [0, 1], [9], *tvd, *tvt, 8, 8).tolist() == \
        [oracle.ST_ID_RANGE]
    assert oracle.consistency([0, 2], [0, 1], [0, 1], [0], *tvd, *tvt, 1, 8).tolist() == \
        [oracle.ST_TOO_LONG]


def test_dpos_hist_on_the_fig2_path():
    g = json.load(open(os.path.join(HERE, "golden", "fig2_example.json")))
    D, T = g["draft_tokens"], g["target_tokens"]
    pairs = []
    for dt, tt in g["path_tokens"]:
        pairs.append([D.index(dt), T.index(tt)])
    path = np.array(pairs, np.int32)
    # hand count: |0-0|, |1-0|, |2-1|, |3-2|, |3-3|
    h = oracle.dpos_hist([0, 4], [0, 4], path, [len(pairs)], np.zeros(4, np.int32), 0, 4)
    assert h.tolist() == [2, 3, 0, 0]
    # map: i*(j) = largest i in column j -> 1, 2, 3, 3; deviations 1, 1, 1, 0
    mp = np.array([1, 2, 3, 3], np.int32)
    h = oracle.dpos_hist([0, 4], [0, 4], path, [len(pairs)], mp, 1, 4)
    assert h.tolist() == [1, 3, 0, 0]
    # overflow bin, accumulation, failed requests add nothing
    h2 = oracle.dpos_hist([0, 4, 8], [0, 4, 8], np.concatenate([path, path]), [5, 0],
                          np.concatenate([mp, mp]), 0, 2, hist=h[:2].copy())
    assert h2.tolist() == [1 + 2, 3 + 3]
