"""GPU parity: the CUDA path through the C ABI against the CPU oracle on the
same seeded inputs, for the five workloads at reduced batch sizes, the
standalone entry points, and the edge cases of the method."""
import numpy as np
import pytest
import torch

import oracle
import paper_2510_15545_gb300 as tt
from paper_2510_15545_gb300 import workload as W

from _parity import TOL, compare, gpu_step, oracle_step, to_np

pytestmark = pytest.mark.gpu
_CACHE = {}


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.skip("needs a GPU")
    tt.load(build_if_missing=True)


def _wl(name, B, seed=0):
    return W.make_workload(name, B=B, seed=seed, vocab_cache=_CACHE)


# ------------------------------------------------------------- whole step

@pytest.mark.parametrize("name,B,seed", [
    ("b1_g4_v32k", 1, 0), ("b1_g4_v32k", 6, 1), ("b64_g8_v152k", 12, 0),
    ("b256_g16_v152k_bf16", 6, 0), ("dtw_4096x64", 24, 0), ("b1024_g8_v201k_bf16", 6, 0)])
def test_step_matches_oracle(name, B, seed):
    wl = _wl(name, B, seed)
    g = gpu_step(wl)
    o = oracle_step(wl)
    c = compare(wl, g, o)
    print(name, c)


@pytest.mark.parametrize("window", [0, 1, 3, -1])
def test_step_other_windows(window):
    wl = _wl("b64_g8_v152k", 8, 5)
    c = compare(wl, gpu_step(wl, window=window), oracle_step(wl, window=window))
    print(window, c)


def test_step_temperatures_and_seed():
    wl = _wl("b256_g16_v152k_bf16", 4, 3)
    kw = dict(temp_draft=0.7, temp_target=0.6, seed=99)
    compare(wl, gpu_step(wl, **kw), oracle_step(wl, **kw))


def test_step_with_draft_probabilities():
    wl = _wl("b64_g8_v152k", 6, 2)
    rng = np.random.default_rng(0)
    probs = rng.uniform(0.01, 0.9, size=wl.n_draft).astype(np.float32)
    g = gpu_step(wl, draft_probs=probs)
    o = oracle_step(wl, draft_probs=probs)
    compare(wl, g, o)


def test_step_request_base_moves_the_uniforms():
    wl = _wl("b64_g8_v152k", 8, 4)
    g = gpu_step(wl, request_base=1000)
    o = oracle_step(wl, request_base=1000)
    compare(wl, g, o)


# ------------------------------------------------- standalone entry points

def _inputs(wl):
    return tt.device_inputs(wl, "cuda")


def test_align_matches_oracle_all_windows():
    wl = _wl("dtw_4096x64", 16, 3)
    inp = _inputs(wl)
    for w in (0, 2, 8, 40, -1):
        prm = inp["params"]
        prm.window = w
        g = to_np(tt.tt_align(inp["batch"], inp["vd"], inp["vt"], prm))
        torch.cuda.synchronize()
        o = oracle.align(wl.draft_off, wl.draft_ids, wl.target_off, wl.target_ids, wl.vd.blob,
                         wl.vd.off, wl.vt.blob, wl.vt.off, w)
        assert np.array_equal(g["status"], o["status"])
        assert np.array_equal(g["path_len"], o["path_len"])
        assert np.array_equal(g["cost"], o["cost"])
        assert np.array_equal(g["map"], o["map"])
        for b in range(wl.B):
            p0 = int(wl.draft_off[b] + wl.target_off[b])
            L = int(o["path_len"][b])
            assert np.array_equal(g["path"][2 * p0:2 * (p0 + L)], o["path"][p0:p0 + L].ravel())


def _random_pairs(rng, B, kmax, mmax, vocab_sz, max_len, empty_ok=False):
    strings = set()
    while len(strings) < vocab_sz:
        n = int(rng.integers(0 if empty_ok else 1, max_len + 1))
        strings.add(bytes(rng.choice(list(b"abcd\x00\xff"), size=n).astype(np.uint8)))
    voc = W.Vocab.from_strings(sorted(strings))
    ks = rng.integers(1, kmax + 1, size=B)
    ms = rng.integers(1, mmax + 1, size=B)
    d_off = np.concatenate([[0], np.cumsum(ks)]).astype(np.int32)
    t_off = np.concatenate([[0], np.cumsum(ms)]).astype(np.int32)
    d_ids = rng.integers(0, vocab_sz, size=int(d_off[-1])).astype(np.int32)
    t_ids = rng.integers(0, vocab_sz, size=int(t_off[-1])).astype(np.int32)
    return voc, d_off, d_ids, t_off, t_ids


@pytest.mark.parametrize("max_len,kmax,mmax,nvoc", [(8, 9, 13, 300), (24, 6, 6, 300),
                                                    (3, 70, 40, 150), (8, 1, 1, 300),
                                                    (3, 256, 512, 150), (256, 4, 4, 60)])
def test_align_random_pairs_and_token_lengths(max_len, kmax, mmax, nvoc):
    """Random byte strings (zero and 0xff bytes, empty strings, tokens longer
    than 8 bytes take the plain dynamic program), random k and m with
    |k - m| often above the window; the largest tile (256 x 512 tokens with no
    band); tokens up to 256 bytes, whose distances can reach 255 and more (the
    one-byte cost tile's escape, recomputed in the sweep)."""
    rng = np.random.default_rng(max_len * 100 + kmax)
    voc, d_off, d_ids, t_off, t_ids = _random_pairs(rng, 40, kmax, mmax, nvoc, max_len,
                                                    empty_ok=True)
    batch = tt.Batch.from_host(d_off, d_ids, t_off, t_ids, device="cuda")
    vt = tt.VocabTable.from_host(voc.blob, voc.off, "cuda")
    for w in (0, 1, 4, -1):
        g = to_np(tt.tt_align(batch, vt, vt, tt.Params(window=w)))
        o = oracle.align(d_off, d_ids, t_off, t_ids, voc.blob, voc.off, voc.blob, voc.off, w)
        for key in ("status", "path_len", "cost", "map"):
            assert np.array_equal(g[key], o[key]), (key, w)
        nd, nt = int(d_off[-1]), int(t_off[-1])
        for b in range(40):
            p0 = int(d_off[b] + t_off[b])
            L = int(o["path_len"][b])
            assert np.array_equal(g["path"][2 * p0:2 * (p0 + L)], o["path"][p0:p0 + L].ravel())


def test_align_status_codes():
    voc = W.Vocab.from_strings([b"a", b"b", b"x" * 300, b"abc"])
    d_off = np.array([0, 1, 1, 2, 3, 4, 5, 7], np.int32)
    d_ids = np.array([0, 0, 9, 0, 3, 1, 1], np.int32)
    t_off = np.array([0, 1, 2, 2, 3, 4, 5, 6], np.int32)
    t_ids = np.array([1, 0, 1, 2, -1, 3], np.int32)
    batch = tt.Batch.from_host(d_off, d_ids, t_off, t_ids, device="cuda")
    v = tt.VocabTable.from_host(voc.blob, voc.off, "cuda")
    g = to_np(tt.tt_align(batch, v, v, tt.Params()))
    o = oracle.align(d_off, d_ids, t_off, t_ids, voc.blob, voc.off, voc.blob, voc.off, 8)
    assert np.array_equal(g["status"], o["status"]), (g["status"], o["status"])
    assert list(g["status"]) == [0, 4, 4, 1, 2, 1, 0]


@pytest.mark.parametrize("dtype", [torch.float32, torch.bfloat16])
@pytest.mark.parametrize("V", [77, 1000, 8192, 8193, 20001])
def test_transfer_and_verify_ragged_widths(dtype, V):
    """Standalone transfer and verify on widths that are not multiples of the
    vector width or the chunk, with temperatures."""
    rng = np.random.default_rng(V)
    B, k = 7, 5
    ms = rng.integers(1, 9, size=B)
    d_off = np.arange(0, B * k + 1, k, dtype=np.int32)
    t_off = np.concatenate([[0], np.cumsum(ms)]).astype(np.int32)
    nd, nt = int(d_off[-1]), int(t_off[-1])
    gen = torch.Generator().manual_seed(V)
    dl = (torch.randn((nd, V), generator=gen) * 2.5).to(dtype)
    tl = (torch.randn((nt + B, V), generator=gen) * 2.5).to(dtype)
    # rows start on 16-byte boundaries (the row pass's contract): pad the stride
    pad = -V % 8

    def padded(x):
        st = torch.full((x.shape[0], V + pad), float("nan"), dtype=dtype, device="cuda")
        st[:, :V] = x.cuda()
        return st[:, :V]
    d_cols = rng.integers(0, V, size=nd).astype(np.int32)
    t_cols = rng.integers(0, V, size=nt).astype(np.int32)
    mp = np.concatenate([np.sort(rng.integers(0, k, size=m)) for m in ms]).astype(np.int32)
    batch = tt.Batch.from_host(d_off, d_cols, t_off, t_cols, device="cuda")
    prm = tt.Params(temp_draft=0.8, temp_target=1.3, seed=7)
    mp_d = torch.as_tensor(mp, device="cuda")
    gt = to_np(tt.tt_transfer(batch, mp_d, prm, draft_logits=padded(dl)))
    ot = oracle.transfer(d_off, d_cols, t_off, mp, dl, 0.8)
    assert np.array_equal(gt["status"], ot["status"])
    assert np.max(np.abs(gt["q_hat"][:nt] - ot["q_hat"])) <= TOL
    q = torch.as_tensor(gt["q_hat"][:nt], device="cuda")
    gv = to_np(tt.tt_verify(batch, q, padded(tl), prm))
    ov = oracle.verify(t_off, t_cols, gt["q_hat"][:nt].astype(np.float64), tl, temp_target=1.3,
                       seed=7)
    g = dict(gv, _target_off=t_off, _draft_off=d_off)

    class _W:
        target_off, draft_off = t_off, d_off
    compare(_W, g, ov, check_align=False, check_q=False)


def test_verify_full_q_matches_oracle():
    wl = W.homogeneous_workload(64, 4, 300, seed=3)
    c = compare(wl, gpu_step(wl, full_q=True, window=8), oracle_step(wl, full_q=True, window=8))
    print(c)


def test_verify_status_codes():
    V = 64
    t_off = np.array([0, 2, 2, 3, 5], np.int32)
    t_cols = np.array([1, 70, 3, 4, 5], np.int32)
    batch = tt.Batch.from_host(np.array([0, 1, 2, 3, 4], np.int32), np.zeros(4, np.int32),
                               t_off, t_cols, device="cuda")
    tl = torch.randn((5 + 4, V))
    q = np.full(5, 0.3)
    gv = to_np(tt.tt_verify(batch, torch.as_tensor(q, dtype=torch.float32, device="cuda"),
                            tl.cuda(), tt.Params()))
    ov = oracle.verify(t_off, t_cols, q, tl)
    assert np.array_equal(gv["status"], ov["status"]), (gv["status"], ov["status"])
    assert list(gv["status"]) == [1, 4, 0, 0]


# -------------------------------------------------- sampling guarantee (GPU)

def test_gpu_emits_the_target_distribution():
    """Alg. 4 losslessness through the CUDA path: homogeneous vocabulary,
    full-q residual, drafts drawn from q; the first emitted token ~ p."""
    from scipy import stats
    V, N = 16, 200000
    rng = np.random.default_rng(8)
    p = rng.dirichlet(np.ones(V) * 0.8)
    q = rng.dirichlet(np.ones(V) * 0.8)
    zp = torch.as_tensor(np.log(p), dtype=torch.float32)
    zq = torch.as_tensor(np.log(q), dtype=torch.float32)
    p32 = torch.softmax(zp.double(), 0).numpy()
    q32 = torch.softmax(zq.double(), 0).numpy()
    t = rng.choice(V, size=N, p=q32).astype(np.int32)
    off = np.arange(N + 1, dtype=np.int32)
    strings = [bytes([65 + i]) for i in range(V)]
    voc = W.Vocab.from_strings(strings)
    batch = tt.Batch.from_host(off, t, off, t, device="cuda")
    vt = tt.VocabTable.from_host(voc.blob, voc.off, "cuda")
    dl = zq.expand(N, V).contiguous().cuda()
    tl = torch.empty((2 * N, V))
    tl[0::2] = zp
    tl[1::2] = zp
    out = to_np(tt.tt_step(batch, vt, vt, dl, tl.cuda(), tt.Params(full_q=True, seed=31)))
    assert np.all(out["status"] == 0)
    first = np.where(out["accepted"] == 1, t, out["next_token"])
    counts = np.bincount(first, minlength=V)
    assert stats.chisquare(counts, p32 * N).pvalue > 1e-4
    assert stats.chisquare(np.bincount(t, minlength=V), p32 * N).pvalue < 1e-6
