"""Seeded synthetic inputs for the TokenTiming verification path.

This module is shared by the tests, the benchmark and the CPU oracle's callers.
It holds none of the method's arithmetic: no token distance, no warping, no
softmax, no accept rule and no random-number generator of the method. It only
builds what the method consumes (§4, Alg. 2 inputs):

* byte-string vocabularies for the draft and the target model (each token id
  names a UTF-8 byte string; App. A / the fragmented-tokenization study treat
  tokens as byte strings),
* draft token ids ``D`` and proxy target ids ``T = encode_t(decode_d(D))``
  (App. A.1, Lemma 1: both spell the same byte string),
* draft and target logits rows (row i of a request's draft block is the
  distribution ``d_i`` was drawn from; target rows ``0..m`` are the m+1
  verification rows of Alg. 2 / Alg. 4, the last one the bonus row).

Real tokenizers, model weights and Spec-Bench are not available, so every
input is synthetic; the shapes follow the five workloads the build is measured
on (batch, draft length, re-encoded length range, vocabulary sizes, logits
dtype and value distribution).

Draft ids are drawn from their own draft rows with the Gumbel-max trick
(``argmax(z / T + G)``), which samples the softmax without evaluating it.
Re-encoding is greedy longest match over the target table (the configs' stated
tokenizer stand-in); the DTW-dominant workload uses a greedy segmentation that
is constrained to hit an exact drawn target length.
"""
from __future__ import annotations

import dataclasses
import math
from typing import Dict, List, Optional, Sequence

import numpy as np
import torch

# Symbols of the synthetic "language": letters, a space and a little
# punctuation, drawn with Zipf(1) frequencies so that short substrings repeat
# the way sub-words do in real text.
_ALPHABET = np.frombuffer(b"etaoinshrdlcumwfgypbvkjxqz .,'-_", dtype=np.uint8)
_ALPHA_W = 1.0 / np.arange(1, len(_ALPHABET) + 1, dtype=np.float64)
_ALPHA_W /= _ALPHA_W.sum()
# Lengths 2..8 of multi-byte tokens (single bytes are ids 0..255).
_LEN_VALUES = np.arange(2, 9)
_LEN_W = np.array([0.10, 0.20, 0.22, 0.18, 0.13, 0.10, 0.07])
MAX_TOKEN_BYTES = 8


@dataclasses.dataclass
class Vocab:
    """A byte-string table: token ``id`` spells ``blob[off[id]:off[id+1]]``."""

    blob: np.ndarray  # uint8
    off: np.ndarray  # int64 [V+1]
    strings: List[bytes]
    index: Dict[bytes, int]

    @property
    def n_tokens(self) -> int:
        return len(self.strings)

    @staticmethod
    def from_strings(strings: Sequence[bytes]) -> "Vocab":
        strings = list(strings)
        lens = np.fromiter((len(s) for s in strings), dtype=np.int64, count=len(strings))
        off = np.zeros(len(strings) + 1, dtype=np.int64)
        np.cumsum(lens, out=off[1:])
        blob = np.frombuffer(b"".join(strings), dtype=np.uint8).copy()
        if blob.size == 0:
            blob = np.zeros(1, dtype=np.uint8)
        index = {s: i for i, s in enumerate(strings)}
        return Vocab(blob=blob, off=off, strings=strings, index=index)


def _random_strings(rng: np.random.Generator, n: int, exclude: set) -> List[bytes]:
    """``n`` distinct multi-byte strings over the alphabet, none in ``exclude``."""
    out: List[bytes] = []
    seen = set(exclude)
    while len(out) < n:
        want = int((n - len(out)) * 1.3) + 64
        lens = rng.choice(_LEN_VALUES, size=want, p=_LEN_W)
        sym = _ALPHABET[rng.choice(len(_ALPHABET), size=(want, MAX_TOKEN_BYTES), p=_ALPHA_W)]
        for row, ln in zip(sym, lens):
            s = row[:ln].tobytes()
            if s not in seen:
                seen.add(s)
                out.append(s)
                if len(out) == n:
                    break
    return out


def make_vocab_pair(V_d: int, V_t: int, seed: int, share: float) -> tuple:
    """Draft and target tables. Ids 0..255 are the 256 single bytes in both
    tables (so greedy re-encoding always succeeds); a fraction ``share`` of the
    draft's multi-byte strings also appear in the target table, the rest of the
    target table is fresh strings."""
    assert V_d > 256 and V_t > 256
    rng = np.random.default_rng(seed)
    singles = [bytes([c]) for c in range(256)]
    d_multi = _random_strings(rng, V_d - 256, set(singles))
    n_shared = min(int(round(share * len(d_multi))), V_t - 256)
    shared_idx = rng.choice(len(d_multi), size=n_shared, replace=False)
    shared = [d_multi[i] for i in shared_idx]
    fresh = _random_strings(rng, V_t - 256 - n_shared, set(singles) | set(d_multi))
    t_multi = shared + fresh
    perm = rng.permutation(len(t_multi))
    t_multi = [t_multi[i] for i in perm]
    return Vocab.from_strings(singles + d_multi), Vocab.from_strings(singles + t_multi)


def greedy_encode(data: bytes, table: Dict[bytes, int]) -> List[int]:
    """Greedy longest-match encoding of ``data`` with ``table`` (the tokenizer
    stand-in named by the workload configs)."""
    out: List[int] = []
    p, n = 0, len(data)
    while p < n:
        for ln in range(min(MAX_TOKEN_BYTES, n - p), 0, -1):
            tid = table.get(data[p:p + ln])
            if tid is not None:
                out.append(tid)
                p += ln
                break
        else:  # unreachable while all single bytes are tokens
            raise ValueError("byte not covered by the table")
    return out


def segment_exact(data: bytes, table: Dict[bytes, int], m: int) -> Optional[List[int]]:
    """Encode ``data`` with exactly ``m`` tokens of ``table``, taking the longest
    admissible piece at each position; ``None`` if no such encoding exists."""
    n = len(data)
    # reach[p]: bit r set iff data[p:] splits into exactly r tokens.
    reach = [0] * (n + 1)
    reach[n] = 1
    for p in range(n - 1, -1, -1):
        acc = 0
        for ln in range(1, min(MAX_TOKEN_BYTES, n - p) + 1):
            if data[p:p + ln] in table:
                acc |= reach[p + ln] << 1
        reach[p] = acc
    if not (reach[0] >> m) & 1:
        return None
    out: List[int] = []
    p, r = 0, m
    while p < n:
        for ln in range(min(MAX_TOKEN_BYTES, n - p), 0, -1):
            tid = table.get(data[p:p + ln])
            if tid is not None and (reach[p + ln] >> (r - 1)) & 1:
                out.append(tid)
                p += ln
                r -= 1
                break
    return out


@dataclasses.dataclass
class WorkloadSpec:
    name: str
    B: int
    k: int
    m_lo: int
    m_hi: int
    V_d: int
    V_t: int
    dtype: torch.dtype
    logits: str  # "normal3" | "zipf"
    zipf_s: float = 1.0
    noise: float = 0.0
    corr_frac: float = 0.0
    corr_rho: float = 0.0
    corr_shift: float = 0.0  # correlated rows: target-only columns lowered by this (nats)
    verify_V: Optional[int] = None  # width of the logits rows if smaller than the vocab
    exact_m: bool = False  # target length drawn uniformly, exact segmentation
    share: float = 0.85
    window: int = 8
    temp_draft: float = 1.0
    temp_target: float = 1.0
    seed: int = 1234  # Philox seed of the method


SPECS: Dict[str, WorkloadSpec] = {
    "b1_g4_v32k": WorkloadSpec("b1_g4_v32k", B=1, k=4, m_lo=3, m_hi=6, V_d=32000, V_t=32768,
                               dtype=torch.float32, logits="normal3", corr_frac=1.0,
                               corr_rho=0.9, corr_shift=3.0),
    "b64_g8_v152k": WorkloadSpec("b64_g8_v152k", B=64, k=8, m_lo=5, m_hi=12, V_d=32000,
                                 V_t=151936, dtype=torch.float32, logits="zipf", zipf_s=1.1,
                                 noise=0.5, corr_frac=1.0, corr_rho=0.9, corr_shift=3.0),
    "b256_g16_v152k_bf16": WorkloadSpec("b256_g16_v152k_bf16", B=256, k=16, m_lo=10, m_hi=24,
                                        V_d=128256, V_t=151936, dtype=torch.bfloat16,
                                        logits="zipf", zipf_s=1.2, noise=1.0, corr_frac=1.0,
                                        corr_rho=0.9, corr_shift=3.0),
    "dtw_4096x64": WorkloadSpec("dtw_4096x64", B=4096, k=64, m_lo=48, m_hi=96, V_d=32000,
                                V_t=151936, dtype=torch.float32, logits="zipf", zipf_s=1.1,
                                noise=0.5, verify_V=4096, exact_m=True),
    "b1024_g8_v201k_bf16": WorkloadSpec("b1024_g8_v201k_bf16", B=1024, k=8, m_lo=5, m_hi=14,
                                        V_d=151936, V_t=201088, dtype=torch.bfloat16,
                                        logits="zipf", zipf_s=1.0, noise=1.0, corr_frac=1.0,
                                        corr_rho=0.9, corr_shift=3.0),
}
# Order of the five workloads (smallest first).
SPEC_ORDER = ["b1_g4_v32k", "b64_g8_v152k", "b256_g16_v152k_bf16", "dtw_4096x64",
              "b1024_g8_v201k_bf16"]


@dataclasses.dataclass
class Workload:
    spec: WorkloadSpec
    vd: Vocab
    vt: Vocab
    draft_off: np.ndarray  # int32 [B+1]
    draft_ids: np.ndarray  # int32 [n_draft]
    target_off: np.ndarray  # int32 [B+1]
    target_ids: np.ndarray  # int32 [n_target]
    draft_cols: np.ndarray  # int32 [n_draft]: column of d_i in its logits row
    target_cols: np.ndarray  # int32 [n_target]
    draft_logits: torch.Tensor  # [n_draft, V_dl]
    target_logits: torch.Tensor  # [n_target + B, V_tl]
    # repetition-penalty histories (logits columns, CSR per request); None = none
    hist_off_d: Optional[np.ndarray] = None
    hist_cols_d: Optional[np.ndarray] = None
    hist_off_t: Optional[np.ndarray] = None
    hist_cols_t: Optional[np.ndarray] = None

    @property
    def B(self) -> int:
        return len(self.draft_off) - 1

    @property
    def n_draft(self) -> int:
        return int(self.draft_off[-1])

    @property
    def n_target(self) -> int:
        return int(self.target_off[-1])

    @property
    def max_k(self) -> int:
        return int(np.diff(self.draft_off).max(initial=0))

    @property
    def max_m(self) -> int:
        return int(np.diff(self.target_off).max(initial=0))

    def subset(self, idx) -> "Workload":
        """Requests ``idx`` as a workload of their own (logits copied to the CPU)."""
        idx = [int(b) for b in idx]
        d_rows, t_rows, d_ids, t_ids, d_cols, t_cols = [], [], [], [], [], []
        d_off, t_off = [0], [0]
        for b in idx:
            d0, d1 = int(self.draft_off[b]), int(self.draft_off[b + 1])
            o0, o1 = int(self.target_off[b]), int(self.target_off[b + 1])
            d_rows.extend(range(d0, d1))
            t_rows.extend(range(o0 + b, o1 + b + 1))
            d_ids.append(self.draft_ids[d0:d1])
            d_cols.append(self.draft_cols[d0:d1])
            t_ids.append(self.target_ids[o0:o1])
            t_cols.append(self.target_cols[o0:o1])
            d_off.append(d_off[-1] + d1 - d0)
            t_off.append(t_off[-1] + o1 - o0)

        def cat(xs):
            return np.concatenate(xs).astype(np.int32) if xs else np.zeros(0, np.int32)
        dl = self.draft_logits[torch.as_tensor(d_rows, device=self.draft_logits.device)].cpu()
        tl = self.target_logits[torch.as_tensor(t_rows, device=self.target_logits.device)].cpu()

        def hist(off, cols):
            if off is None:
                return None, None
            parts = [cols[off[b]:off[b + 1]] for b in idx]
            o = np.concatenate([[0], np.cumsum([len(x) for x in parts])]).astype(np.int32)
            return o, cat(parts)
        hod, hcd = hist(self.hist_off_d, self.hist_cols_d)
        hot, hct = hist(self.hist_off_t, self.hist_cols_t)
        return dataclasses.replace(self, draft_off=np.array(d_off, np.int32),
                                   target_off=np.array(t_off, np.int32), draft_ids=cat(d_ids),
                                   target_ids=cat(t_ids), draft_cols=cat(d_cols),
                                   target_cols=cat(t_cols), draft_logits=dl, target_logits=tl,
                                   hist_off_d=hod, hist_cols_d=hcd, hist_off_t=hot,
                                   hist_cols_t=hct)

    def request(self, b: int) -> dict:
        d0, d1 = int(self.draft_off[b]), int(self.draft_off[b + 1])
        t0, t1 = int(self.target_off[b]), int(self.target_off[b + 1])
        return dict(draft_ids=self.draft_ids[d0:d1], target_ids=self.target_ids[t0:t1],
                    draft_rows=(d0, d1), target_rows=(t0 + b, t1 + b + 1))


# ---------------------------------------------------------------------------
# logits

def _affine_perm_ranks(gen: torch.Generator, R: int, V: int, device) -> torch.Tensor:
    """1-based ranks under a random affine permutation x -> (a x + c) mod V per
    row (a coprime to V): a cheap stand-in for an independent random
    permutation of the vocabulary in every row."""
    a = torch.randint(1, V, (R,), generator=gen, device=device, dtype=torch.int64).cpu().numpy()
    bad = np.gcd(a, V) != 1
    while bad.any():  # step to the next candidate; 1 is always coprime
        a[bad] = a[bad] % (V - 1) + 1
        bad = np.gcd(a, V) != 1
    a = torch.from_numpy(a)
    c = torch.randint(0, V, (R,), generator=gen, device=device, dtype=torch.int64).cpu()
    x = torch.arange(V, device=device, dtype=torch.int64)
    return ((x[None, :] * a.to(device)[:, None] + c.to(device)[:, None]) % V) + 1


def _gen_rows(spec: WorkloadSpec, R: int, V: int, gen: torch.Generator, device) -> torch.Tensor:
    """``R`` fp32 logits rows of width ``V`` following the workload's recipe."""
    out = torch.empty((R, V), dtype=torch.float32, device=device)
    step = max(1, (1 << 26) // max(V, 1))
    for r0 in range(0, R, step):
        r1 = min(R, r0 + step)
        n = r1 - r0
        if spec.logits == "normal3":
            blk = torch.randn((n, V), generator=gen, device=device) * 3.0
        else:
            ranks = _affine_perm_ranks(gen, n, V, device).to(torch.float32)
            blk = -spec.zipf_s * torch.log(ranks)
            if spec.noise:
                blk += torch.randn((n, V), generator=gen, device=device) * spec.noise
        out[r0:r1] = blk
    return out


def _gumbel_argmax(rows: torch.Tensor, temp: float, gen: torch.Generator) -> torch.Tensor:
    """Draws one index per row from softmax(rows / temp) by the Gumbel-max trick."""
    u = torch.rand(rows.shape, generator=gen, device=rows.device, dtype=torch.float32)
    u = u.clamp_(min=1e-20)
    g = -torch.log(-torch.log(u))
    return torch.argmax(rows.float() / temp + g, dim=1)


def make_workload(name: str, *, B: Optional[int] = None, seed: int = 0,
                  device: str = "cpu", vocab_cache: Optional[dict] = None) -> Workload:
    """Builds a seeded workload. ``B`` overrides the batch (reduced test sizes);
    logits are created directly on ``device``."""
    spec = SPECS[name]
    B = spec.B if B is None else B
    key = (spec.V_d, spec.V_t, spec.share)
    if vocab_cache is not None and key in vocab_cache:
        vd, vt = vocab_cache[key]
    else:
        vd, vt = make_vocab_pair(spec.V_d, spec.V_t, seed=1000 + spec.V_d + spec.V_t,
                                 share=spec.share)
        if vocab_cache is not None:
            vocab_cache[key] = (vd, vt)
    rng = np.random.default_rng(seed)
    gen = torch.Generator(device=device)
    gen.manual_seed(seed * 7919 + 17)
    V_dl = spec.verify_V or spec.V_d
    V_tl = spec.verify_V or spec.V_t
    k = spec.k

    draft_ids = np.zeros((B, k), dtype=np.int64)
    target_lists: List[List[int]] = []
    if spec.exact_m:
        # The text S is a run of random multi-byte target tokens; D splits S into
        # exactly k draft tokens and T into exactly the drawn m target tokens
        # (both spell S, Lemma 1), each taking the longest admissible pieces.
        pool = np.arange(256, vt.n_tokens)
        m_goal = rng.integers(spec.m_lo, spec.m_hi + 1, size=B)
        for b in range(B):
            for _ in range(1000):
                words = pool[rng.integers(0, len(pool), size=int(rng.integers(34, 42)))]
                data = b"".join(vt.strings[i] for i in words)
                d = segment_exact(data, vd.index, k)
                t = segment_exact(data, vt.index, int(m_goal[b])) if d is not None else None
                if t is not None:
                    break
            else:
                raise RuntimeError("could not reach the drawn target length")
            draft_ids[b] = d
            target_lists.append(t)
        draft_logits = _gen_rows(spec, B * k, V_dl, gen, device)
    else:
        draft_logits = _gen_rows(spec, B * k, V_dl, gen, device)
        pending = np.arange(B)
        for _ in range(400):
            rows = draft_logits.view(B, k, V_dl)[torch.as_tensor(pending, device=device)]
            ids = _gumbel_argmax(rows.reshape(-1, V_dl), spec.temp_draft, gen)
            ids = ids.view(len(pending), k).cpu().numpy()
            still = []
            for n_, b in enumerate(pending):
                data = b"".join(vd.strings[i] for i in ids[n_])
                t = greedy_encode(data, vt.index)
                if spec.m_lo <= len(t) <= spec.m_hi:
                    draft_ids[b] = ids[n_]
                    while len(target_lists) <= b:
                        target_lists.append([])
                    target_lists[b] = t
                else:
                    still.append(b)
            pending = np.array(still, dtype=np.int64)
            if len(pending) == 0:
                break
        else:
            raise RuntimeError("re-encoded lengths did not land in range")
    m_arr = np.array([len(t) for t in target_lists], dtype=np.int64)
    draft_off = np.arange(0, B * k + 1, k, dtype=np.int32)
    target_off = np.zeros(B + 1, dtype=np.int32)
    np.cumsum(m_arr, out=target_off[1:])
    n_target = int(target_off[-1])
    target_ids = np.concatenate([np.asarray(t, dtype=np.int32) for t in target_lists]) \
        if n_target else np.zeros(0, dtype=np.int32)
    draft_ids_flat = draft_ids.reshape(-1).astype(np.int32)

    target_logits = _gen_rows(spec, n_target + B, V_tl, gen, device)
    if spec.corr_frac > 0:
        _correlate(spec, target_logits, draft_logits, draft_off, target_off, draft_ids_flat,
                   target_ids, vd, vt, rng, device)

    if spec.verify_V:
        draft_cols = (draft_ids_flat % spec.verify_V).astype(np.int32)
        target_cols = (target_ids % spec.verify_V).astype(np.int32)
    else:
        draft_cols = draft_ids_flat.copy()
        target_cols = target_ids.copy()
    return Workload(spec=spec, vd=vd, vt=vt, draft_off=draft_off, draft_ids=draft_ids_flat,
                    target_off=target_off, target_ids=target_ids, draft_cols=draft_cols,
                    target_cols=target_cols,
                    draft_logits=draft_logits.to(spec.dtype),
                    target_logits=target_logits.to(spec.dtype))


def _source_rows(vd, vt, d_ids, t_ids) -> np.ndarray:
    """For each target token, the draft token holding its last byte (tokenizer
    bookkeeping of the re-encoding, not an alignment)."""
    ends = np.cumsum([len(vd.strings[i]) for i in d_ids])
    t_ends = np.cumsum([len(vt.strings[i]) for i in t_ids])
    return np.searchsorted(ends, t_ends - 1, side="right").clip(max=len(d_ids) - 1)


def _correlate(spec, target_logits, draft_logits, draft_off, target_off, draft_ids, target_ids,
               vd, vt, rng, device):
    """Makes the target rows of a fraction ``corr_frac`` of the requests
    correlated (coefficient ``corr_rho``) with the draft row holding the same
    bytes, through the injection that sends a target string to the draft id
    spelling it: z_t = rho * z_d + sqrt(1 - rho^2) * sd(z_d) * N(0, 1) on the
    columns the two vocabularies share; the target-only columns of those rows
    are lowered by ``corr_shift``, standing for a target that puts little mass
    on strings the draft cannot spell. The bonus row follows the last draft
    row. Rows are processed in blocks of bounded size."""
    inj = np.full(vt.n_tokens, -1, dtype=np.int64)
    for tid, s in enumerate(vt.strings):
        did = vd.index.get(s)
        if did is not None:
            inj[tid] = did
    have = np.nonzero(inj >= 0)[0]
    have_t = torch.as_tensor(have, device=device)
    from_d = torch.as_tensor(inj[have], device=device)
    rho = spec.corr_rho
    B = len(draft_off) - 1
    gen = torch.Generator(device=device)
    gen.manual_seed(int(rng.integers(0, 2**31)))
    chosen = rng.random(B) < spec.corr_frac
    rows_t, rows_d = [], []
    for b in np.nonzero(chosen)[0]:
        d0, d1 = int(draft_off[b]), int(draft_off[b + 1])
        t0, t1 = int(target_off[b]), int(target_off[b + 1])
        src = _source_rows(vd, vt, draft_ids[d0:d1], target_ids[t0:t1])
        src = np.concatenate([src, [d1 - d0 - 1]])
        rows_t.extend(t0 + int(b) + np.arange(len(src)))
        rows_d.extend(d0 + src.astype(np.int64))
    if not rows_t:
        return
    rows_t = torch.as_tensor(np.asarray(rows_t, dtype=np.int64), device=device)
    rows_d = torch.as_tensor(np.asarray(rows_d, dtype=np.int64), device=device)
    step = max(1, (1 << 26) // max(target_logits.shape[1], 1))
    for r0 in range(0, len(rows_t), step):
        rt, rd = rows_t[r0:r0 + step], rows_d[r0:r0 + step]
        zd = draft_logits[rd][:, from_d]
        sd = zd.std(dim=1, keepdim=True)
        noise = torch.randn(zd.shape, generator=gen, device=device) * sd
        blk = target_logits[rt]
        if spec.corr_shift:
            blk -= spec.corr_shift
        blk[:, have_t] = rho * zd + math.sqrt(1 - rho * rho) * noise
        target_logits[rt] = blk


def homogeneous_workload(B: int, k: int, V: int, *, seed: int = 0, device: str = "cpu",
                         logit_scale: float = 1.5, target_noise: float = 0.5,
                         dtype=torch.float32) -> Workload:
    """Standard speculative decoding as a special case (Alg. 4): draft and target
    share one table of V single-token strings, T = D, and the draft ids are drawn
    from the draft rows. Target rows are the draft rows plus noise, so acceptance
    is frequent but not certain."""
    strings = [bytes([65 + (i % 26), 97 + (i // 26) % 26, 48 + (i // 676) % 10]) for i in range(V)]
    voc = Vocab.from_strings(strings)
    gen = torch.Generator(device=device)
    gen.manual_seed(seed * 104729 + 5)
    draft_logits = torch.randn((B * k, V), generator=gen, device=device) * logit_scale
    ids = _gumbel_argmax(draft_logits, 1.0, gen).cpu().numpy().astype(np.int32)
    draft_off = np.arange(0, B * k + 1, k, dtype=np.int32)
    target_off = draft_off.copy()
    tl = torch.empty((B * (k + 1), V), dtype=torch.float32, device=device)
    dl3 = draft_logits.view(B, k, V)
    tl3 = tl.view(B, k + 1, V)
    tl3[:, :k] = dl3 + target_noise * torch.randn((B, k, V), generator=gen, device=device)
    tl3[:, k] = torch.randn((B, V), generator=gen, device=device) * logit_scale
    spec = WorkloadSpec("homogeneous", B=B, k=k, m_lo=k, m_hi=k, V_d=V, V_t=V,
                        dtype=dtype, logits="normal")
    return Workload(spec=spec, vd=voc, vt=voc, draft_off=draft_off, draft_ids=ids,
                    target_off=target_off, target_ids=ids.copy(), draft_cols=ids.copy(),
                    target_cols=ids.copy(), draft_logits=draft_logits.to(dtype),
                    target_logits=tl.to(dtype))


def with_histories(wl: Workload, lo: int, hi: int, seed: int = 0) -> Workload:
    """The workload with seeded repetition-penalty histories: each request gets
    between lo and hi earlier tokens per family (logits columns), half of them
    drawn from the request's own rows by the Gumbel-max trick (tokens the rows
    make likely, as a real context's tokens are) and half uniformly, with
    repeats allowed."""
    rng = np.random.default_rng(seed * 7919 + 17)
    gen = torch.Generator(device=wl.target_logits.device)
    gen.manual_seed(seed * 104729 + 23)

    def family(off_rows, logits, extra_row):
        offs, cols = [0], []
        V = logits.shape[1]
        for b in range(wl.B):
            n = int(rng.integers(lo, hi + 1))
            r0, r1 = int(off_rows[b]) + (b if extra_row else 0), int(off_rows[b + 1]) + (
                b + 1 if extra_row else 0)
            n_like = n // 2
            if n_like > 0 and r1 > r0:
                rows = torch.as_tensor(rng.integers(r0, r1, size=n_like), device=logits.device)
                u = torch.rand((n_like, V), generator=gen, device=logits.device).clamp_(1e-12, 1)
                g = logits[rows].float() - torch.log(-torch.log(u))
                like = g.argmax(1).cpu().numpy().astype(np.int32)
            else:
                like = np.zeros(0, np.int32)
            uni = rng.integers(0, V, size=n - len(like)).astype(np.int32)
            h = np.concatenate([like, uni])
            rng.shuffle(h)
            cols.append(h)
            offs.append(offs[-1] + len(h))
        return np.array(offs, np.int32), (np.concatenate(cols).astype(np.int32) if cols
                                          else np.zeros(0, np.int32))
    hod, hcd = family(wl.draft_off, wl.draft_logits, False)
    hot, hct = family(wl.target_off, wl.target_logits, True)
    return dataclasses.replace(wl, hist_off_d=hod, hist_cols_d=hcd, hist_off_t=hot,
                               hist_cols_t=hct)
