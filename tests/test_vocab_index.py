"""The re-encoding index built on the host by tt_vocab_index_build (no GPU):
every prefix of every non-empty token has exactly one slot, a whole token's
slot names the smallest id of its string, and nothing else is stored. The slot
keys are re-derived here from the layout the library documents (bytes up to 8,
then a chained fingerprint with MurmurHash3's finaliser)."""
import numpy as np

from paper_2510_15545_gb300 import binding
from paper_2510_15545_gb300 import workload as W

M64 = (1 << 64) - 1


def fmix64(x):
    x ^= x >> 33
    x = (x * 0xff51afd7ed558ccd) & M64
    x ^= x >> 33
    x = (x * 0xc4ceb9fe1a85ec53) & M64
    x ^= x >> 33
    return x


def key_of(s):
    key = 0
    for L, byte in enumerate(s, 1):
        if L <= 8:
            key |= byte << (8 * (L - 1))
        else:
            key = fmix64((key + byte * 0x9e3779b97f4a7c15 + L) & M64)
    return key


def build(strings):
    voc = W.Vocab.from_strings(strings)
    L = binding.load()
    n = L.tt_vocab_index_bytes(len(strings), int(voc.off[-1]))
    host = np.zeros(n, np.uint8)
    off = np.ascontiguousarray(voc.off, np.int64)
    blob = np.ascontiguousarray(voc.blob, np.uint8)
    code = L.tt_vocab_index_build(blob.ctypes.data if blob.size else None, off.ctypes.data,
                                  len(strings), host.ctypes.data, n)
    return code, host


def test_index_holds_every_prefix_once():
    rng = np.random.default_rng(3)
    strings = []
    for _ in range(400):
        L = int(rng.integers(1, 20))
        strings.append(bytes(rng.choice(list(b"abc\x00"), L).astype(np.uint8).tolist()))
    strings += strings[:25]  # repeated strings
    strings.append(b"")      # an empty token is left out
    code, host = build(strings)
    assert code == 0
    hdr = host[:16].view(np.int32)
    n_slots, max_len, n_tokens = int(hdr[1]), int(hdr[2]), int(hdr[3])
    assert n_slots & (n_slots - 1) == 0 and max_len == max(len(s) for s in strings)
    assert n_tokens == len(strings)
    slots = host[64:64 + 16 * n_slots]
    keys = slots.view(np.uint64)[0::2]
    lens = slots.view(np.int32)[2::4]
    ids = slots.view(np.int32)[3::4]
    got = {}
    for s in range(n_slots):
        if lens[s]:
            k = (int(keys[s]), int(lens[s]))
            assert k not in got
            got[k] = int(ids[s])
    want = {}
    for v, s in enumerate(strings):
        for L in range(1, len(s) + 1):
            k = (key_of(s[:L]), L)
            cur = want.get(k, -1)
            if L == len(s):
                want[k] = v if cur < 0 else min(cur, v)
            else:
                want.setdefault(k, -1)
    assert got == want
    assert 2 * len(got) <= n_slots


def test_index_rejects_too_long_tokens():
    code, _ = build([b"a", b"x" * 257])
    assert code == binding.TT_ERR_UNSUPPORTED
