"""GPU parity of the re-encoding, the Lemma-1 check and the delta-pos histogram
(tt_encode, tt_consistency, tt_dpos_hist through the C ABI) against the oracle:
bit-exact tokens, offsets, statuses and counts."""
import numpy as np
import pytest
import torch

import oracle
import paper_2510_15545_gb300 as tt
from paper_2510_15545_gb300 import workload as W

pytestmark = pytest.mark.gpu
_CACHE = {}


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.skip("needs a GPU")
    tt.load(build_if_missing=True)


def _dev(x, dtype=torch.int32):
    return torch.as_tensor(np.asarray(x), dtype=dtype, device="cuda")


def gpu_encode(d_off, d_ids, vd, vt, max_m, capacity=None, index=None):
    vdt = tt.VocabTable.from_host(vd.blob, vd.off, "cuda")
    vtt = tt.VocabTable.from_host(vt.blob, vt.off, "cuda")
    idx = index if index is not None else tt.vocab_index(vt.blob, vt.off)
    d_ids = np.asarray(d_ids, np.int32)
    ids = _dev(d_ids if d_ids.size else np.zeros(1, np.int32))
    r = tt.tt_encode(_dev(d_off), ids, vdt, vtt, idx, max_m, capacity=capacity)
    torch.cuda.synchronize()
    off = r["target_off"].cpu().numpy()
    return dict(target_off=off, target_ids=r["target_ids"].cpu().numpy()[:off[-1]],
                status=r["status"].cpu().numpy()[:len(d_off) - 1])


def check(g, o):
    assert np.array_equal(g["status"], o["status"])
    assert np.array_equal(g["target_off"], o["target_off"])
    assert np.array_equal(g["target_ids"], o["target_ids"])


@pytest.mark.parametrize("name,B", [("b1_g4_v32k", 1), ("b64_g8_v152k", 64),
                                    ("b256_g16_v152k_bf16", 96), ("dtw_4096x64", 64),
                                    ("b1024_g8_v201k_bf16", 128)])
def test_encode_matches_oracle_on_the_workloads(name, B):
    wl = W.make_workload(name, B=B, seed=2, vocab_cache=_CACHE)
    g = gpu_encode(wl.draft_off, wl.draft_ids, wl.vd, wl.vt, 512)
    o = oracle.encode(wl.draft_off, wl.draft_ids, wl.vd.blob, wl.vd.off, wl.vt.blob, wl.vt.off,
                      512)
    check(g, o)
    assert (g["status"] == 0).all()


def rand_vocab(rng, n, max_len, alphabet, all_bytes=True, dup=0):
    out = [bytes([i]) for i in range(256)] if all_bytes else []
    seen = set(out)
    for _ in range(50 * n):  # small alphabets and lengths run out of strings
        if len(out) >= n:
            break
        L = int(rng.integers(1, max_len + 1))
        s = bytes(rng.choice(list(alphabet), L).astype(np.uint8).tolist())
        if s not in seen:
            seen.add(s)
            out.append(s)
    for _ in range(dup):  # repeated strings: the smallest id must win
        out.append(out[int(rng.integers(0, len(out)))])
    return W.Vocab.from_strings(out)


@pytest.mark.parametrize("max_len", [4, 8, 9, 20, 64])
def test_encode_random_vocabularies(max_len):
    """Tokens up to 64 bytes (fingerprint keys past 8 bytes), repeated strings,
    zero and 0xff bytes, empty draft tokens, ragged batches."""
    rng = np.random.default_rng(max_len)
    alphabet = b"ab\x00\xff"
    vd = rand_vocab(rng, 500, max_len, alphabet)
    vd = W.Vocab.from_strings(vd.strings + [b""])  # an empty draft token
    vt = rand_vocab(rng, 700, max_len, alphabet, dup=30)
    B = 150
    ks = rng.integers(0, 40, B)
    d_off = np.concatenate([[0], np.cumsum(ks)]).astype(np.int32)
    d_ids = rng.integers(0, len(vd.strings), int(d_off[-1])).astype(np.int32)
    for max_m in (512, 7):
        g = gpu_encode(d_off, d_ids, vd, vt, max_m)
        o = oracle.encode(d_off, d_ids, vd.blob, vd.off, vt.blob, vt.off, max_m)
        check(g, o)
    assert (o["status"] == oracle.ST_TOO_LONG).any() and (o["status"] == 0).any()
    # a capacity that cuts the batch short
    cap = int(o["target_off"][-1]) // 2
    g = gpu_encode(d_off, d_ids, vd, vt, 7, capacity=cap)
    check(g, oracle.encode(d_off, d_ids, vd.blob, vd.off, vt.blob, vt.off, 7, capacity=cap))


def test_encode_status_codes():
    vd = W.Vocab.from_strings([b"abc", b"z", b"q" * 300, b"x" * 7])
    vt = W.Vocab.from_strings([b"a", b"b", b"c", b"bc", b"q", b"x"])
    # ok, no match (z), empty, id out of range, too long (> 2048 bytes), bad offsets
    d_off = np.array([0, 1, 2, 2, 3, 12, 13, 12], np.int32)
    d_ids = np.array([0, 1, 9] + [2] * 9 + [3], np.int32)
    g = gpu_encode(d_off, d_ids, vd, vt, 512)
    o = oracle.encode(d_off, d_ids, vd.blob, vd.off, vt.blob, vt.off, 512)
    check(g, o)
    assert o["status"].tolist() == [0, oracle.ST_NO_MATCH, oracle.ST_EMPTY, oracle.ST_ID_RANGE,
                                    oracle.ST_TOO_LONG, 0, oracle.ST_BAD_OFFSETS]


def test_encode_index_can_be_reused_and_empty_batch():
    wl = W.make_workload("b64_g8_v152k", B=16, seed=5, vocab_cache=_CACHE)
    idx = tt.vocab_index(wl.vt.blob, wl.vt.off)
    o = oracle.encode(wl.draft_off, wl.draft_ids, wl.vd.blob, wl.vd.off, wl.vt.blob, wl.vt.off, 64)
    for _ in range(2):
        check(gpu_encode(wl.draft_off, wl.draft_ids, wl.vd, wl.vt, 64, index=idx), o)
    g = gpu_encode(np.zeros(1, np.int32), [], wl.vd, wl.vt, 64, index=idx)
    assert g["target_off"].tolist() == [0]


def _batch(d_off, d_ids, t_off, t_ids):
    return tt.Batch.from_host(d_off, d_ids, t_off, t_ids, device="cuda")


def test_consistency_matches_oracle():
    wl = W.make_workload("b256_g16_v152k_bf16", B=64, seed=4, vocab_cache=_CACHE)
    vd = tt.VocabTable.from_host(wl.vd.blob, wl.vd.off, "cuda")
    vt = tt.VocabTable.from_host(wl.vt.blob, wl.vt.off, "cuda")
    rng = np.random.default_rng(0)
    t_ids = wl.target_ids.copy()
    # perturb some requests: swap in a random token, drop the last token
    for b in range(0, wl.B, 5):
        t0, t1 = int(wl.target_off[b]), int(wl.target_off[b + 1])
        t_ids[t0 + int(rng.integers(0, t1 - t0))] = int(rng.integers(0, len(wl.vt.strings)))
    t_off = wl.target_off.copy()
    t_off[wl.B] -= 1  # the last request loses its last token
    for max_k, max_m in ((256, 512), (8, 512)):
        batch = tt.Batch.from_host(wl.draft_off, wl.draft_ids, t_off, t_ids, device="cuda",
                                   max_k=max_k, max_m=max_m)
        g = tt.tt_consistency(batch, vd, vt).cpu().numpy()[:wl.B]
        o = oracle.consistency(wl.draft_off, wl.draft_ids, t_off, t_ids, wl.vd.blob, wl.vd.off,
                               wl.vt.blob, wl.vt.off, max_k, max_m)
        assert np.array_equal(g, o)
        if max_k == 256:
            assert (o == oracle.ST_INCONSISTENT).sum() >= wl.B // 5 and (o == 0).any()
        else:
            assert (o == oracle.ST_TOO_LONG).all()
    batch = tt.Batch.from_host(wl.draft_off, wl.draft_ids, wl.target_off, wl.target_ids,
                               device="cuda")
    assert (tt.tt_consistency(batch, vd, vt).cpu().numpy()[:wl.B] == 0).all()  # Lemma 1


def test_consistency_of_the_gpu_encoding():
    wl = W.make_workload("b1024_g8_v201k_bf16", B=64, seed=1, vocab_cache=_CACHE)
    g = gpu_encode(wl.draft_off, wl.draft_ids, wl.vd, wl.vt, 512)
    batch = tt.Batch.from_host(wl.draft_off, wl.draft_ids, g["target_off"],
                               g["target_ids"], device="cuda")
    vd = tt.VocabTable.from_host(wl.vd.blob, wl.vd.off, "cuda")
    vt = tt.VocabTable.from_host(wl.vt.blob, wl.vt.off, "cuda")
    assert (tt.tt_consistency(batch, vd, vt).cpu().numpy()[:wl.B] == 0).all()


@pytest.mark.parametrize("w", [-1, 8, 2])
def test_dpos_hist_matches_oracle(w):
    wl = W.make_workload("dtw_4096x64", B=48, seed=6, vocab_cache=_CACHE)
    inp = tt.device_inputs(wl, "cuda")
    prm = inp["params"]
    prm.window = w
    al = tt.tt_align(inp["batch"], inp["vd"], inp["vt"], prm)
    o = oracle.align(wl.draft_off, wl.draft_ids, wl.target_off, wl.target_ids, wl.vd.blob,
                     wl.vd.off, wl.vt.blob, wl.vt.off, w)
    path = al["path"].cpu().numpy()
    for mode in (0, 1):
        for n_bins in (1, 5, 200):
            g = tt.tt_dpos_hist(inp["batch"], al["path"], al["path_len"], al["map"], mode,
                                n_bins).cpu().numpy()
            want = oracle.dpos_hist(wl.draft_off, wl.target_off, o["path"], o["path_len"],
                                    o["map"], mode, n_bins)
            assert np.array_equal(g, want), (mode, n_bins)
            # the same counts from the GPU's own path and map
            assert np.array_equal(g, oracle.dpos_hist(wl.draft_off, wl.target_off, path,
                                                      al["path_len"].cpu().numpy(),
                                                      al["map"].cpu().numpy(), mode, n_bins))
    # accumulation over calls
    h = torch.zeros(16, dtype=torch.int64, device="cuda")
    tt.tt_dpos_hist(inp["batch"], al["path"], al["path_len"], al["map"], 0, 16, hist=h)
    tt.tt_dpos_hist(inp["batch"], al["path"], al["path_len"], al["map"], 0, 16, hist=h)
    one = oracle.dpos_hist(wl.draft_off, wl.target_off, o["path"], o["path_len"], o["map"], 0, 16)
    assert np.array_equal(h.cpu().numpy(), 2 * one)
