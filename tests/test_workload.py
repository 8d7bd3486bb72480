"""The synthetic inputs keep the properties the method relies on: the proxy
target ids spell the same bytes as the draft ids (App. A.1, Lemma 1), lengths
land in each workload's range, and generation is deterministic per seed."""
import numpy as np
import pytest

from paper_2510_15545_gb300 import workload as W


@pytest.fixture(scope="module")
def cache():
    return {}


@pytest.mark.parametrize("name,B", [("b1_g4_v32k", 8), ("b64_g8_v152k", 8), ("dtw_4096x64", 6),
                                    ("b256_g16_v152k_bf16", 4), ("b1024_g8_v201k_bf16", 4)])
def test_lemma1_and_ranges(name, B, cache):
    wl = W.make_workload(name, B=B, seed=3, vocab_cache=cache)
    spec = wl.spec
    assert wl.B == B and wl.n_draft == B * spec.k
    for b in range(B):
        r = wl.request(b)
        s_d = b"".join(wl.vd.strings[i] for i in r["draft_ids"])
        s_t = b"".join(wl.vt.strings[i] for i in r["target_ids"])
        assert s_d == s_t
        assert spec.m_lo <= len(r["target_ids"]) <= spec.m_hi
    assert wl.draft_logits.shape == (wl.n_draft, spec.verify_V or spec.V_d)
    assert wl.target_logits.shape == (wl.n_target + B, spec.verify_V or spec.V_t)
    assert wl.draft_logits.dtype == spec.dtype
    assert int(wl.draft_cols.max()) < wl.draft_logits.shape[1]
    assert int(wl.target_cols.max()) < wl.target_logits.shape[1]
    tok_len = np.diff(wl.vt.off)
    assert tok_len.min() >= 1 and tok_len.max() <= 8


def test_deterministic(cache):
    a = W.make_workload("b1_g4_v32k", B=4, seed=9, vocab_cache=cache)
    b = W.make_workload("b1_g4_v32k", B=4, seed=9, vocab_cache=cache)
    assert np.array_equal(a.target_ids, b.target_ids)
    assert bool((a.target_logits == b.target_logits).all())


def test_greedy_encode_is_longest_match():
    table = {bytes([c]): c for c in range(256)}
    table.update({b"ab": 300, b"abc": 301, b"cd": 302})
    assert W.greedy_encode(b"abcd", table) == [301, ord("d")]
    assert W.segment_exact(b"abcd", table, 2) == [301, ord("d")]
    assert W.segment_exact(b"abcd", table, 3) == [300, ord("c"), ord("d")]
    assert W.segment_exact(b"abcd", table, 5) is None
