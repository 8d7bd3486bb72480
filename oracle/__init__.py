"""CPU oracle of the TokenTiming verification path (test infrastructure).

Only the tests, ``__graft_entry__.smoke()`` and the benchmark's CPU-baseline and
reference legs import this package. The product path (the CUDA library and its
binding) never does; the two share no code.

``build()`` compiles ``tto.c`` with gcc into ``libtto.so`` beside it; the
wrappers below marshal numpy arrays (or CPU torch tensors for logits) into the
C entry points and return numpy results.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
from typing import Optional

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "tto.c")
_LIB = os.path.join(_HERE, "libtto.so")
_lib = None


class _Pen(ctypes.Structure):
    """tto_penalty: the repetition penalty of one family (tto.h)."""
    _fields_ = [("hist_off", ctypes.c_void_p), ("hist_cols", ctypes.c_void_p),
                ("theta", ctypes.c_float)]

# Status bits (shared meaning with the CUDA library, defined independently).
ST_ID_RANGE, ST_TOO_LONG, ST_EMPTY, ST_BAD_OFFSETS = 1, 2, 4, 8
ST_NO_MATCH, ST_INCONSISTENT = 128, 256


def build(force: bool = False) -> str:
    """Compiles the oracle (plain C, -O2, no fast-math) if it is missing or stale."""
    stale = (not os.path.exists(_LIB)
             or os.path.getmtime(_LIB) < max(os.path.getmtime(_SRC),
                                              os.path.getmtime(os.path.join(_HERE, "tto.h"))))
    if force or stale:
        tmp = _LIB + ".tmp%d" % os.getpid()
        subprocess.check_call(["gcc", "-std=c11", "-O2", "-fPIC", "-shared", "-fno-fast-math",
                               "-ffp-contract=off", "-o", tmp, _SRC, "-lm"])
        os.replace(tmp, _LIB)
    return _LIB


def lib():
    global _lib
    if _lib is None:
        build()
        L = ctypes.CDLL(_LIB)
        P = ctypes.c_void_p
        i32, i64, u64, f64 = ctypes.c_int32, ctypes.c_int64, ctypes.c_uint64, ctypes.c_double
        L.tto_lev.argtypes = [P, i32, P, i32]
        L.tto_lev.restype = i32
        L.tto_dtw.argtypes = [i32, i32, P, i32, P, P]
        L.tto_dtw.restype = i64
        L.tto_philox4x64_10.argtypes = [P, P, P]
        L.tto_philox4x64_10.restype = None
        L.tto_uniform.argtypes = [u64, u64, u64, u64]
        L.tto_uniform.restype = f64
        L.tto_softmax.argtypes = [P, i32, i64, f64, P]
        L.tto_softmax.restype = None
        L.tto_logsumexp.argtypes = [P, i32, i64, f64]
        L.tto_logsumexp.restype = f64
        L.tto_align.argtypes = [i32, P, P, P, P, P, P, i32, P, P, i32, i32, P, P, P, P, P]
        L.tto_align.restype = None
        L.tto_transfer.argtypes = [i32, P, P, P, P, P, i32, i64, i32, P, f64, P, P]
        L.tto_transfer.restype = None
        L.tto_verify.argtypes = [i32, P, P, P, P, i32, i64, i32, f64, P, P, P, i32, i64, i32,
                                 f64, i32, u64, u64, P, P, P, P, P, P]
        L.tto_verify.restype = None
        L.tto_filtered_probs.argtypes = [P, i32, i64, f64, i32, f64, P, P]
        L.tto_filtered_probs.restype = f64
        L.tto_transfer2.argtypes = [i32, P, P, P, P, P, i32, i64, i32, P, f64, i32, f64, P, P, P]
        L.tto_transfer2.restype = None
        L.tto_verify2.argtypes = [i32, P, P, P, P, i32, i64, i32, f64, P, P, P, i32, i64, i32,
                                  f64, i32, u64, u64, i32, f64, i32, f64, P, P, P, P, P, P]
        L.tto_verify2.restype = None
        L.tto_transfer3.argtypes = [i32, P, P, P, P, P, i32, i64, i32, P, f64, i32, f64, P, P, P,
                                    P]
        L.tto_transfer3.restype = None
        L.tto_verify3.argtypes = [i32, P, P, P, P, i32, i64, i32, f64, P, P, P, i32, i64, i32,
                                  f64, i32, u64, u64, i32, f64, i32, f64, P, P, P, P, P, P, P, P,
                                  P]
        L.tto_verify3.restype = None
        L.tto_transfer_pen.argtypes = [i32, P, P, P, P, P, i32, i64, i32, P, f64, i32, f64, P, P,
                                       P, P, P]
        L.tto_transfer_pen.restype = None
        L.tto_verify_pen.argtypes = [i32, P, P, P, P, i32, i64, i32, f64, P, P, P, i32, i64, i32,
                                     f64, i32, u64, u64, i32, f64, i32, f64, P, P, P, P, P, P, P,
                                     P, P, P]
        L.tto_verify_pen.restype = None
        L.tto_encode.argtypes = [i32, P, P, P, P, i32, P, P, i32, i32, i32, i32, P, P, P]
        L.tto_encode.restype = None
        L.tto_consistency.argtypes = [i32, P, P, P, P, P, P, i32, P, P, i32, i32, i32, P]
        L.tto_consistency.restype = None
        L.tto_dpos_hist.argtypes = [i32, P, P, P, P, P, i32, i32, P]
        L.tto_dpos_hist.restype = None
        _lib = L
    return _lib


def _p(a) -> Optional[int]:
    return None if a is None else a.ctypes.data


def _i32(a):
    return np.ascontiguousarray(a, dtype=np.int32)


def _logits(x):
    """(buffer, dtype code, row stride, V) for fp32 / bf16 rows given as a CPU
    torch tensor or a float32 numpy array."""
    if isinstance(x, np.ndarray):
        x = np.ascontiguousarray(x, dtype=np.float32)
        return x, 0, x.shape[1], x.shape[1]
    import torch
    t = x.detach().cpu().contiguous()
    if t.dtype == torch.float32:
        return t.numpy(), 0, t.shape[1], t.shape[1]
    if t.dtype == torch.bfloat16:
        return t.view(torch.int16).numpy(), 1, t.shape[1], t.shape[1]
    raise TypeError("logits must be float32 or bfloat16")


def lev(s: bytes, t: bytes) -> int:
    a = np.frombuffer(s, dtype=np.uint8) if s else np.zeros(1, np.uint8)
    b = np.frombuffer(t, dtype=np.uint8) if t else np.zeros(1, np.uint8)
    return int(lib().tto_lev(_p(a), len(s), _p(b), len(t)))


def dtw(d: np.ndarray, w: int):
    """Alg. 1 on a k x m integer cost matrix -> (C*, path as list of (i, j))."""
    d = np.ascontiguousarray(d, dtype=np.int32)
    k, m = d.shape
    path = np.zeros(2 * (k + m) + 2, dtype=np.int32)
    L = np.zeros(1, dtype=np.int32)
    c = lib().tto_dtw(k, m, _p(d), int(w), _p(path), _p(L))
    n = int(L[0])
    return int(c), [(int(path[2 * x]), int(path[2 * x + 1])) for x in range(n)]


def philox4x64_10(ctr, key):
    c = np.asarray(ctr, dtype=np.uint64)
    k = np.asarray(key, dtype=np.uint64)
    out = np.zeros(4, dtype=np.uint64)
    lib().tto_philox4x64_10(_p(c), _p(k), _p(out))
    return [int(v) for v in out]


def uniform(seed: int, pos: int, stream: int, request: int) -> float:
    return float(lib().tto_uniform(seed, pos, stream, request))


def softmax(row, T: float = 1.0) -> np.ndarray:
    buf, dt, _, V = _logits(row.reshape(1, -1) if hasattr(row, "reshape") else row)
    out = np.zeros(V, dtype=np.float64)
    lib().tto_softmax(_p(buf), dt, V, float(T), _p(out))
    return out


def logsumexp(row, T: float = 1.0) -> float:
    buf, dt, _, V = _logits(row.reshape(1, -1))
    return float(lib().tto_logsumexp(_p(buf), dt, V, float(T)))


def align(draft_off, draft_ids, target_off, target_ids, vd_blob, vd_off, vt_blob, vt_off,
          w: int) -> dict:
    draft_off, draft_ids = _i32(draft_off), _i32(draft_ids)
    target_off, target_ids = _i32(target_off), _i32(target_ids)
    vd_blob = np.ascontiguousarray(vd_blob, dtype=np.uint8)
    vt_blob = np.ascontiguousarray(vt_blob, dtype=np.uint8)
    vd_off = np.ascontiguousarray(vd_off, dtype=np.int64)
    vt_off = np.ascontiguousarray(vt_off, dtype=np.int64)
    B = len(draft_off) - 1
    nd, nt = max(int(draft_off[-1]), 0), max(int(target_off[-1]), 0)
    path = np.full(2 * (nd + nt) + 2, -1, dtype=np.int32)
    path_len = np.zeros(B, np.int32)
    cost = np.zeros(B, np.int32)
    mp = np.full(max(nt, 1), -1, dtype=np.int32)
    status = np.zeros(B, np.int32)
    lib().tto_align(B, _p(draft_off), _p(draft_ids), _p(target_off), _p(target_ids),
                    _p(vd_blob), _p(vd_off), len(vd_off) - 1, _p(vt_blob), _p(vt_off),
                    len(vt_off) - 1, int(w), _p(path), _p(path_len), _p(cost), _p(mp),
                    _p(status))
    return dict(path=path[:2 * (nd + nt)].reshape(-1, 2), path_len=path_len, cost=cost,
                map=mp[:nt], status=status)


def filtered_probs(row, temp: float = 1.0, top_k: int = 0, top_p: float = 1.0):
    """Temperature, top-k, top-p distribution of one row (tto_filtered_probs);
    returns (probs over all columns, log-normaliser of the kept set, boundary bits)."""
    buf, dt, stride, V = _logits(row if np.ndim(row) == 2 or not isinstance(row, np.ndarray)
                                 else np.asarray(row, np.float32)[None, :])
    out = np.zeros(V, np.float64)
    bnd = np.zeros(1, np.int32)
    lse = lib().tto_filtered_probs(_p(buf), dt, V, float(temp), int(top_k), float(top_p),
                                   _p(out), _p(bnd))
    return out, lse, int(bnd[0])


def _penalty(theta, hist_off, hist_cols, keep: list):
    """(pointer to a tto_penalty or None) for a family's repetition penalty."""
    if theta is None or float(np.float32(theta)) == 1.0:
        return None
    ho = None if hist_off is None else _i32(hist_off)
    hc = None if hist_cols is None else _i32(hist_cols if len(hist_cols) else np.zeros(1))
    pen = _Pen(_p(ho), _p(hc), float(theta))
    keep += [ho, hc, pen]
    return ctypes.addressof(pen)


def transfer(draft_off, draft_cols, target_off, mp, draft_logits, temp_draft: float = 1.0,
             draft_probs=None, top_k: int = 0, top_p: float = 1.0, rep_penalty: float = 1.0,
             hist_off=None, hist_cols=None) -> dict:
    draft_off, target_off, mp = _i32(draft_off), _i32(target_off), _i32(mp)
    draft_cols = _i32(draft_cols)
    B = len(draft_off) - 1
    nt = max(int(target_off[-1]), 0)
    q = np.zeros(max(nt, 1), dtype=np.float64)
    status = np.zeros(B, np.int32)
    probs = None if draft_probs is None else np.ascontiguousarray(draft_probs, np.float32)
    if draft_logits is not None:
        buf, dt, stride, V = _logits(draft_logits)
    else:
        buf, dt, stride, V = None, 0, 0, 0
    bnd = np.zeros(max(B, 1), np.int32)
    nd = max(int(draft_off[-1]), 0)
    drow = np.zeros(max(nd, 1), np.int32)
    keep = []
    pen = _penalty(rep_penalty, hist_off, hist_cols, keep)
    lib().tto_transfer_pen(B, _p(draft_off), _p(draft_cols), _p(target_off), _p(mp), _p(buf), dt,
                           stride, V, _p(probs), float(temp_draft), int(top_k), float(top_p), pen,
                           _p(q), _p(status), _p(bnd), _p(drow))
    return dict(q_hat=q[:nt], status=status, boundary=bnd[:B], drow_bnd=drow[:nd])


def verify(target_off, target_cols, q_hat, target_logits, *, temp_target: float = 1.0,
           seed: int = 1234, request_base: int = 0, full_q: bool = False, draft_off=None,
           mp=None, draft_logits=None, temp_draft: float = 1.0, top_k_target: int = 0,
           top_p_target: float = 1.0, top_k_draft: int = 0, top_p_draft: float = 1.0,
           rep_penalty_target: float = 1.0, hist_off_t=None, hist_cols_t=None) -> dict:
    target_off, target_cols = _i32(target_off), _i32(target_cols)
    q_hat = np.ascontiguousarray(q_hat, dtype=np.float64)
    B = len(target_off) - 1
    nt = max(int(target_off[-1]), 0)
    tbuf, tdt, tstride, Vt = _logits(target_logits)
    if full_q:
        dbuf, ddt, dstride, Vd = _logits(draft_logits)
        draft_off, mp = _i32(draft_off), _i32(mp)
    else:
        dbuf, ddt, dstride, Vd = None, 0, 0, 0
    acc = np.zeros(B, np.int32)
    nxt = np.zeros(B, np.int32)
    p_hat = np.zeros(max(nt, 1), np.float64)
    lse = np.zeros(nt + B, np.float64)
    status = np.zeros(B, np.int32)
    bnd = np.zeros(B, np.int32)
    row_bnd = np.zeros(max(nt + B, 1), np.int32)
    tok_lo = np.full(max(B, 1), -1, np.int32)
    tok_hi = np.full(max(B, 1), -1, np.int32)
    keep = []
    pen = _penalty(rep_penalty_target, hist_off_t, hist_cols_t, keep)
    lib().tto_verify_pen(B, _p(target_off), _p(target_cols), _p(q_hat), _p(tbuf), tdt, tstride,
                         Vt, float(temp_target), _p(draft_off) if full_q else None,
                         _p(mp) if full_q else None, _p(dbuf), ddt, dstride, Vd,
                         float(temp_draft), int(bool(full_q)), int(seed), int(request_base),
                         int(top_k_target), float(top_p_target), int(top_k_draft),
                         float(top_p_draft), pen, _p(acc), _p(nxt), _p(p_hat), _p(lse),
                         _p(status), _p(bnd), _p(row_bnd), _p(tok_lo), _p(tok_hi))
    return dict(accepted=acc, next_token=nxt, p_hat=p_hat[:nt], lse=lse, status=status,
                boundary=bnd, row_bnd=row_bnd[:nt + B], tok_lo=tok_lo[:B], tok_hi=tok_hi[:B])


def step(wl, *, window: Optional[int] = None, temp_draft: Optional[float] = None,
         temp_target: Optional[float] = None, seed: Optional[int] = None,
         request_base: int = 0, full_q: bool = False, draft_probs=None, top_k_draft: int = 0,
         top_p_draft: float = 1.0, top_k_target: int = 0, top_p_target: float = 1.0,
         rep_penalty_draft: float = 1.0, rep_penalty_target: float = 1.0) -> dict:
    """The whole verification path for a workload (align -> transfer -> verify);
    the repetition penalties use the workload's histories (hist_*_d / hist_*_t)."""
    spec = wl.spec
    window = spec.window if window is None else window
    temp_draft = spec.temp_draft if temp_draft is None else temp_draft
    temp_target = spec.temp_target if temp_target is None else temp_target
    seed = spec.seed if seed is None else seed
    al = align(wl.draft_off, wl.draft_ids, wl.target_off, wl.target_ids, wl.vd.blob, wl.vd.off,
               wl.vt.blob, wl.vt.off, window)
    hist = lambda name: getattr(wl, name, None)
    tr = transfer(wl.draft_off, wl.draft_cols, wl.target_off, al["map"], wl.draft_logits,
                  temp_draft, draft_probs, top_k=top_k_draft, top_p=top_p_draft,
                  rep_penalty=rep_penalty_draft, hist_off=hist("hist_off_d"),
                  hist_cols=hist("hist_cols_d"))
    ve = verify(wl.target_off, wl.target_cols, tr["q_hat"], wl.target_logits,
                temp_target=temp_target, seed=seed, request_base=request_base, full_q=full_q,
                draft_off=wl.draft_off, mp=al["map"], draft_logits=wl.draft_logits,
                temp_draft=temp_draft, top_k_target=top_k_target, top_p_target=top_p_target,
                top_k_draft=top_k_draft, top_p_draft=top_p_draft,
                rep_penalty_target=rep_penalty_target, hist_off_t=hist("hist_off_t"),
                hist_cols_t=hist("hist_cols_t"))
    # the fused step reports the alignment's problems first, else the later stages'
    status = np.where(al["status"] != 0, al["status"], tr["status"] | ve["status"])
    out = dict(al)
    out.update(q_hat=tr["q_hat"], p_hat=ve["p_hat"], lse=ve["lse"], accepted=ve["accepted"],
               next_token=ve["next_token"], boundary=ve["boundary"] | tr["boundary"],
               status=status, row_bnd=ve["row_bnd"], drow_bnd=tr["drow_bnd"],
               tok_lo=ve["tok_lo"], tok_hi=ve["tok_hi"])
    bad = status != 0
    out["accepted"] = np.where(bad, 0, out["accepted"]).astype(np.int32)
    out["next_token"] = np.where(bad, -1, out["next_token"]).astype(np.int32)
    return out


def encode(draft_off, draft_ids, vd_blob, vd_off, vt_blob, vt_off, max_m: int,
           max_bytes: int = 2048, capacity: Optional[int] = None) -> dict:
    """Re-encoding T = encode_t(decode_d(D)) by greedy longest match (tto_encode)."""
    draft_off, draft_ids = _i32(draft_off), _i32(draft_ids)
    vd_blob = np.ascontiguousarray(vd_blob, dtype=np.uint8)
    vt_blob = np.ascontiguousarray(vt_blob, dtype=np.uint8)
    vd_off = np.ascontiguousarray(vd_off, dtype=np.int64)
    vt_off = np.ascontiguousarray(vt_off, dtype=np.int64)
    B = len(draft_off) - 1
    if capacity is None:
        capacity = B * max_m
    target_off = np.zeros(B + 1, np.int32)
    target_ids = np.full(max(capacity, 1), -1, np.int32)
    status = np.zeros(max(B, 1), np.int32)
    lib().tto_encode(B, _p(draft_off), _p(draft_ids), _p(vd_blob), _p(vd_off), len(vd_off) - 1,
                     _p(vt_blob), _p(vt_off), len(vt_off) - 1, int(max_m), int(max_bytes),
                     int(capacity), _p(target_off), _p(target_ids), _p(status))
    return dict(target_off=target_off, target_ids=target_ids[:target_off[-1]], status=status[:B])


def consistency(draft_off, draft_ids, target_off, target_ids, vd_blob, vd_off, vt_blob, vt_off,
                max_k: int, max_m: int) -> np.ndarray:
    """Lemma 1 as a check: status per request (tto_consistency)."""
    draft_off, draft_ids = _i32(draft_off), _i32(draft_ids)
    target_off, target_ids = _i32(target_off), _i32(target_ids)
    vd_blob = np.ascontiguousarray(vd_blob, dtype=np.uint8)
    vt_blob = np.ascontiguousarray(vt_blob, dtype=np.uint8)
    vd_off = np.ascontiguousarray(vd_off, dtype=np.int64)
    vt_off = np.ascontiguousarray(vt_off, dtype=np.int64)
    B = len(draft_off) - 1
    status = np.zeros(max(B, 1), np.int32)
    lib().tto_consistency(B, _p(draft_off), _p(draft_ids), _p(target_off), _p(target_ids),
                          _p(vd_blob), _p(vd_off), len(vd_off) - 1, _p(vt_blob), _p(vt_off),
                          len(vt_off) - 1, int(max_k), int(max_m), _p(status))
    return status[:B]


def dpos_hist(draft_off, target_off, path, path_len, mp, mode: int, n_bins: int,
              hist=None) -> np.ndarray:
    """Delta-pos histogram of the DTW paths (mode 0) or of the map (mode 1)."""
    draft_off, target_off = _i32(draft_off), _i32(target_off)
    path = _i32(np.asarray(path).reshape(-1))
    path_len, mp = _i32(path_len), _i32(mp if len(mp) else np.zeros(1, np.int32))
    out = np.zeros(n_bins, np.int64) if hist is None else np.ascontiguousarray(hist, np.int64)
    lib().tto_dpos_hist(len(draft_off) - 1, _p(draft_off), _p(target_off), _p(path),
                        _p(path_len), _p(mp), int(mode), int(n_bins), _p(out))
    return out
