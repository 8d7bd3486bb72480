"""ctypes binding of libtt.so (include/tt.h): the same entry points, with
PyTorch tensors for device memory and streams. Argument marshalling only --
every step of the verification path runs in the library's CUDA kernels. There
is no fallback: if the library is missing or a call fails, an exception says so.
"""
from __future__ import annotations

import ctypes
import dataclasses
import os
from typing import Optional, Sequence

import numpy as np
import torch

from . import _build

c_i32, c_i64, c_u64, c_f32, c_p = (ctypes.c_int32, ctypes.c_int64, ctypes.c_uint64,
                                   ctypes.c_float, ctypes.c_void_p)

TT_OK, TT_ERR_INVALID_ARG, TT_ERR_UNSUPPORTED, TT_ERR_CUDA = 0, 1, 2, 3
TT_REQ_ID_OUT_OF_RANGE, TT_REQ_TOO_LONG, TT_REQ_EMPTY, TT_REQ_BAD_OFFSETS, TT_REQ_NOT_FINITE = (
    1, 2, 4, 8, 16)
TT_REQ_NO_MATCH, TT_REQ_INCONSISTENT = 128, 256
TT_MAX_ENCODE_BYTES, TT_MAX_DPOS_BINS = 2048, 4096
TT_F32, TT_BF16 = 0, 1
TT_MAX_K, TT_MAX_M, TT_MAX_TOKEN_BYTES = 256, 512, 256


class TTError(RuntimeError):
    def __init__(self, fn: str, code: int, msg: str):
        super().__init__("%s failed: %s (%d)" % (fn, msg, code))
        self.code = code


class _Vocab(ctypes.Structure):
    _fields_ = [("bytes", c_p), ("offsets", c_p), ("n_tokens", c_i32), ("n_bytes", c_i64)]


class _Logits(ctypes.Structure):
    _fields_ = [("data", c_p), ("dtype", c_i32), ("n_cols", c_i32), ("row_stride", c_i64),
                ("n_rows", c_i64)]


class _Shards(ctypes.Structure):
    _fields_ = [("S", c_i32), ("shards", ctypes.POINTER(_Logits)), ("col0", ctypes.POINTER(c_i32))]


class _Params(ctypes.Structure):
    _fields_ = [("window", c_i32), ("temp_draft", c_f32), ("temp_target", c_f32),
                ("full_q", c_i32), ("seed", c_u64), ("request_base", c_u64), ("events", c_p),
                ("top_k_draft", c_i32), ("top_p_draft", c_f32), ("top_k_target", c_i32),
                ("top_p_target", c_f32), ("rep_penalty_draft", c_f32),
                ("rep_penalty_target", c_f32)]


class _Batch(ctypes.Structure):
    _fields_ = [("B", c_i32), ("n_draft", c_i32), ("n_target", c_i32), ("max_k", c_i32),
                ("max_m", c_i32), ("draft_off", c_p), ("draft_ids", c_p), ("draft_cols", c_p),
                ("target_off", c_p), ("target_ids", c_p), ("target_cols", c_p),
                ("hist_off_d", c_p), ("hist_cols_d", c_p), ("hist_off_t", c_p),
                ("hist_cols_t", c_p), ("n_hist_d", c_i32), ("n_hist_t", c_i32)]


class _StepOut(ctypes.Structure):
    _fields_ = [("accepted", c_p), ("next_token", c_p), ("status", c_p), ("path", c_p),
                ("path_len", c_p), ("cost", c_p), ("map", c_p), ("q_hat", c_p), ("p_hat", c_p),
                ("lse", c_p)]


_lib = None
EXPORTS = ("tt_workspace_bytes", "tt_workspace_bytes_for", "tt_align", "tt_transfer", "tt_verify", "tt_step",
           "tt_step_noalloc", "tt_status_string", "tt_last_cuda_error", "tt_version",
           "tt_vocab_index_bytes", "tt_vocab_index_build", "tt_encode_workspace_bytes",
           "tt_encode", "tt_consistency", "tt_dpos_hist", "tt_sharded_workspace_bytes",
           "tt_verify_sharded")
TT_MAX_SHARDS = 8
TT_NOALLOC_SCRATCH_BYTES = 16 << 20


def lib_path() -> str:
    return _build.LIB


def load(build_if_missing: bool = False):
    """Loads libtt.so (building it first when asked and nvcc is present)."""
    global _lib
    if _lib is not None:
        return _lib
    path = lib_path()
    if build_if_missing and (not os.path.exists(path) or _build.is_stale()):
        _build.build()
    if not os.path.exists(path):
        raise RuntimeError("libtt.so is not built (%s); run __graft_entry__.build() or "
                           "python -m paper_2510_15545_gb300._build" % path)
    L = ctypes.CDLL(path)
    P = ctypes.POINTER
    L.tt_workspace_bytes.argtypes = [P(_Batch), c_i32, c_i32]
    L.tt_workspace_bytes.restype = ctypes.c_size_t
    L.tt_workspace_bytes_for.argtypes = [P(_Batch), c_i32, c_i32, P(_Params)]
    L.tt_workspace_bytes_for.restype = ctypes.c_size_t
    L.tt_align.argtypes = [P(_Batch), P(_Vocab), P(_Vocab), P(_Params), c_p, c_p, c_p, c_p, c_p,
                           c_p]
    L.tt_align.restype = c_i32
    L.tt_transfer.argtypes = [P(_Batch), c_p, P(_Logits), c_p, P(_Params), c_p, ctypes.c_size_t,
                              c_p, c_p, c_p]
    L.tt_transfer.restype = c_i32
    L.tt_verify.argtypes = [P(_Batch), c_p, P(_Logits), P(_Logits), c_p, P(_Params), c_p,
                            ctypes.c_size_t, c_p, c_p, c_p, c_p, c_p, c_p]
    L.tt_verify.restype = c_i32
    L.tt_step.argtypes = [P(_Batch), P(_Vocab), P(_Vocab), P(_Logits), c_p, P(_Logits),
                          P(_Params), c_p, ctypes.c_size_t, P(_StepOut), c_p]
    L.tt_step.restype = c_i32
    L.tt_step_noalloc.argtypes = [P(_Batch), P(_Vocab), P(_Vocab), P(_Logits), c_p, P(_Logits),
                                  P(_Params), P(_StepOut), c_p]
    L.tt_step_noalloc.restype = c_i32
    L.tt_sharded_workspace_bytes.argtypes = [P(_Batch), P(_Shards)]
    L.tt_sharded_workspace_bytes.restype = ctypes.c_size_t
    L.tt_verify_sharded.argtypes = [P(_Batch), c_p, P(_Shards), P(_Params), c_p, ctypes.c_size_t,
                                    c_p, c_p, c_p, c_p, c_p, c_p, c_p]
    L.tt_verify_sharded.restype = c_i32
    L.tt_status_string.argtypes = [c_i32]
    L.tt_status_string.restype = ctypes.c_char_p
    L.tt_last_cuda_error.argtypes = []
    L.tt_last_cuda_error.restype = c_i32
    L.tt_version.argtypes = []
    L.tt_version.restype = c_i32
    L.tt_vocab_index_bytes.argtypes = [c_i32, c_i64]
    L.tt_vocab_index_bytes.restype = ctypes.c_size_t
    L.tt_vocab_index_build.argtypes = [c_p, c_p, c_i32, c_p, ctypes.c_size_t]
    L.tt_vocab_index_build.restype = c_i32
    L.tt_encode_workspace_bytes.argtypes = [c_i32, c_i32]
    L.tt_encode_workspace_bytes.restype = ctypes.c_size_t
    L.tt_encode.argtypes = [c_i32, c_i32, c_p, c_p, P(_Vocab), P(_Vocab), c_p, c_i32, c_i32,
                            c_p, c_p, c_p, c_p, ctypes.c_size_t, c_p]
    L.tt_encode.restype = c_i32
    L.tt_consistency.argtypes = [P(_Batch), P(_Vocab), P(_Vocab), c_p, c_p]
    L.tt_consistency.restype = c_i32
    L.tt_dpos_hist.argtypes = [P(_Batch), c_p, c_p, c_p, c_i32, c_i32, c_p, c_p]
    L.tt_dpos_hist.restype = c_i32
    _lib = L
    return L


# --------------------------------------------------------------- arguments

def _ptr(t: Optional[torch.Tensor]) -> Optional[int]:
    if t is None:
        return None
    return t.data_ptr()


@dataclasses.dataclass
class Batch:
    """A CSR batch of requests held in device memory (int32 tensors)."""

    draft_off: torch.Tensor
    draft_ids: torch.Tensor
    target_off: torch.Tensor
    target_ids: torch.Tensor
    draft_cols: Optional[torch.Tensor] = None
    target_cols: Optional[torch.Tensor] = None
    B: int = 0
    n_draft: int = 0
    n_target: int = 0
    max_k: int = 1
    max_m: int = 1
    # repetition-penalty histories (logits columns, CSR per request); None = empty
    hist_off_d: Optional[torch.Tensor] = None
    hist_cols_d: Optional[torch.Tensor] = None
    hist_off_t: Optional[torch.Tensor] = None
    hist_cols_t: Optional[torch.Tensor] = None
    n_hist_d: int = 0
    n_hist_t: int = 0

    def with_history(self, hist_off_d=None, hist_cols_d=None, hist_off_t=None,
                     hist_cols_t=None) -> "Batch":
        """This batch with repetition-penalty histories (host or device arrays)."""
        dev = self.target_off.device

        def d(x):
            return None if x is None else torch.as_tensor(x, dtype=torch.int32).to(dev).contiguous()
        b = dataclasses.replace(self, hist_off_d=d(hist_off_d), hist_cols_d=d(hist_cols_d),
                                hist_off_t=d(hist_off_t), hist_cols_t=d(hist_cols_t))
        b.n_hist_d = 0 if hist_off_d is None else int(np.asarray(hist_off_d)[-1])
        b.n_hist_t = 0 if hist_off_t is None else int(np.asarray(hist_off_t)[-1])
        return b

    @staticmethod
    def from_host(draft_off, draft_ids, target_off, target_ids, draft_cols=None,
                  target_cols=None, device="cuda", max_k=None, max_m=None) -> "Batch":
        def dev(x):
            if x is None:
                return None
            return torch.as_tensor(x, dtype=torch.int32).to(device).contiguous()
        do = torch.as_tensor(draft_off, dtype=torch.int64)
        to = torch.as_tensor(target_off, dtype=torch.int64)
        B = len(do) - 1
        ks = (do[1:] - do[:-1]) if B > 0 else torch.zeros(0, dtype=torch.int64)
        ms = (to[1:] - to[:-1]) if B > 0 else torch.zeros(0, dtype=torch.int64)
        mk = int(ks.max()) if B > 0 else 1
        mm = int(ms.max()) if B > 0 else 1
        return Batch(dev(draft_off), dev(draft_ids), dev(target_off), dev(target_ids),
                     dev(draft_cols), dev(target_cols), B=B,
                     n_draft=int(do[-1]) if B > 0 else 0, n_target=int(to[-1]) if B > 0 else 0,
                     max_k=max(1, min(TT_MAX_K, mk)) if max_k is None else max_k,
                     max_m=max(1, min(TT_MAX_M, mm)) if max_m is None else max_m)

    def _c(self) -> _Batch:
        return _Batch(self.B, self.n_draft, self.n_target, self.max_k, self.max_m,
                      _ptr(self.draft_off), _ptr(self.draft_ids), _ptr(self.draft_cols),
                      _ptr(self.target_off), _ptr(self.target_ids), _ptr(self.target_cols),
                      _ptr(self.hist_off_d), _ptr(self.hist_cols_d), _ptr(self.hist_off_t),
                      _ptr(self.hist_cols_t), int(self.n_hist_d), int(self.n_hist_t))


@dataclasses.dataclass
class VocabTable:
    """Token byte strings in device memory: id v spells bytes[offsets[v]:offsets[v+1]]."""

    bytes: torch.Tensor  # uint8
    offsets: torch.Tensor  # int64 [V+1]

    @staticmethod
    def from_host(blob, offsets, device="cuda") -> "VocabTable":
        b = torch.as_tensor(blob, dtype=torch.uint8)
        if b.numel() == 0:
            b = torch.zeros(1, dtype=torch.uint8)
        return VocabTable(b.to(device).contiguous(),
                          torch.as_tensor(offsets, dtype=torch.int64).to(device).contiguous())

    def _c(self) -> _Vocab:
        return _Vocab(_ptr(self.bytes), _ptr(self.offsets), self.offsets.numel() - 1,
                      self.bytes.numel())


@dataclasses.dataclass
class Params:
    window: int = 8
    temp_draft: float = 1.0
    temp_target: float = 1.0
    full_q: bool = False
    seed: int = 1234
    request_base: int = 0
    events: Optional[Sequence] = None  # 4 torch.cuda.Event (tt_step stage timing)
    # sampling filters (0 / 1.0 = off); top_p < 1 needs top_k >= 1
    top_k_draft: int = 0
    top_p_draft: float = 1.0
    top_k_target: int = 0
    top_p_target: float = 1.0
    # repetition penalty per family (1.0 = off); needs that family's top_k >= 1
    rep_penalty_draft: float = 1.0
    rep_penalty_target: float = 1.0

    def _c(self, keep: list) -> _Params:
        ev = None
        if self.events is not None:
            arr = (c_p * 4)(*[e.cuda_event for e in self.events])
            keep.append(arr)
            ev = ctypes.cast(arr, c_p)
        return _Params(int(self.window), float(self.temp_draft), float(self.temp_target),
                       int(bool(self.full_q)), int(self.seed), int(self.request_base), ev,
                       int(self.top_k_draft), float(self.top_p_draft), int(self.top_k_target),
                       float(self.top_p_target), float(self.rep_penalty_draft),
                       float(self.rep_penalty_target))


def _logits(t: Optional[torch.Tensor]) -> Optional[_Logits]:
    if t is None:
        return None
    if t.dim() != 2 or t.stride(1) != 1:
        raise ValueError("logits must be a 2-D tensor with unit column stride")
    if t.dtype == torch.float32:
        dt = TT_F32
    elif t.dtype == torch.bfloat16:
        dt = TT_BF16
    else:
        raise TypeError("logits must be float32 or bfloat16")
    return _Logits(t.data_ptr(), dt, t.shape[1], t.stride(0), t.shape[0])


def _stream(stream) -> Optional[int]:
    if stream is None:
        return torch.cuda.current_stream().cuda_stream
    return stream.cuda_stream if hasattr(stream, "cuda_stream") else int(stream)


def _check(fn: str, code: int):
    if code != TT_OK:
        msg = load().tt_status_string(code).decode()
        if code == TT_ERR_CUDA:
            msg += " (cudaError %d)" % load().tt_last_cuda_error()
        raise TTError(fn, code, msg)


def _empty(n, dtype, device):
    return torch.empty(max(int(n), 1), dtype=dtype, device=device)


# ----------------------------------------------------------- entry points

def tt_workspace_bytes(batch: Batch, V_d: int, V_t: int,
                       params: Optional["Params"] = None) -> int:
    if params is None:
        return int(load().tt_workspace_bytes(ctypes.byref(batch._c()), int(V_d), int(V_t)))
    return int(load().tt_workspace_bytes_for(ctypes.byref(batch._c()), int(V_d), int(V_t),
                                             ctypes.byref(params._c([]))))


def workspace(batch: Batch, V_d: int, V_t: int, device="cuda",
              params: Optional["Params"] = None) -> torch.Tensor:
    """Scratch for transfer / verify / step (the caching allocator aligns to 512 bytes);
    pass the call's params when it uses sampling filters."""
    return torch.empty(max(tt_workspace_bytes(batch, V_d, V_t, params), 256), dtype=torch.uint8,
                       device=device)


class AlignCall:
    """A prepared tt_align call: the ctypes argument blocks and the output
    pointers are built once, so a repeated alignment costs one foreign call."""

    def __init__(self, batch: Batch, vd: VocabTable, vt: VocabTable, params: Params, *,
                 out=None, stream=None):
        dev = batch.draft_off.device
        o = dict(out or {})
        o.setdefault("path", _empty(2 * (batch.n_draft + batch.n_target), torch.int32, dev))
        o.setdefault("path_len", _empty(batch.B, torch.int32, dev))
        o.setdefault("cost", _empty(batch.B, torch.int32, dev))
        o.setdefault("map", _empty(batch.n_target, torch.int32, dev))
        o.setdefault("status", _empty(batch.B, torch.int32, dev))
        self.out = o
        self._keep = [batch, vd, vt, o]
        self._b = batch._c()
        self._vd = vd._c()
        self._vt = vt._c()
        self._prm = params._c(self._keep)
        self._ptrs = [_ptr(o[k]) for k in ("path", "path_len", "cost", "map", "status")]
        self._stream = _stream(stream)
        self._lib = load()

    def __call__(self) -> dict:
        code = self._lib.tt_align(ctypes.byref(self._b), ctypes.byref(self._vd),
                                  ctypes.byref(self._vt), ctypes.byref(self._prm), *self._ptrs,
                                  self._stream)
        _check("tt_align", code)
        return self.out


def tt_align(batch: Batch, vd: VocabTable, vt: VocabTable, params: Params, *, out=None,
             stream=None) -> dict:
    return AlignCall(batch, vd, vt, params, out=out, stream=stream)()


def tt_transfer(batch: Batch, map: torch.Tensor, params: Params, *, draft_logits=None,
                draft_probs=None, ws=None, out=None, stream=None) -> dict:
    dev = batch.draft_off.device
    o = dict(out or {})
    o.setdefault("q_hat", _empty(batch.n_target, torch.float32, dev))
    o.setdefault("status", _empty(batch.B, torch.int32, dev))
    if ws is None and draft_logits is not None:
        ws = workspace(batch, draft_logits.shape[1], 0, dev, params)
    keep = []
    L = _logits(draft_logits)
    code = load().tt_transfer(ctypes.byref(batch._c()), _ptr(map),
                              ctypes.byref(L) if L is not None else None, _ptr(draft_probs),
                              ctypes.byref(params._c(keep)), _ptr(ws),
                              0 if ws is None else ws.numel(), _ptr(o["q_hat"]),
                              _ptr(o["status"]), _stream(stream))
    _check("tt_transfer", code)
    return o


def tt_verify(batch: Batch, q_hat: torch.Tensor, target_logits: torch.Tensor, params: Params, *,
              draft_logits=None, map=None, ws=None, out=None, stream=None) -> dict:
    dev = batch.target_off.device
    o = dict(out or {})
    o.setdefault("accepted", _empty(batch.B, torch.int32, dev))
    o.setdefault("next_token", _empty(batch.B, torch.int32, dev))
    o.setdefault("status", _empty(batch.B, torch.int32, dev))
    o.setdefault("p_hat", _empty(batch.n_target, torch.float32, dev))
    o.setdefault("lse", _empty(batch.n_target + batch.B, torch.float32, dev))
    if ws is None:
        Vd = draft_logits.shape[1] if (params.full_q and draft_logits is not None) else 0
        ws = workspace(batch, Vd, target_logits.shape[1], dev, params)
    keep = []
    Lt, Ld = _logits(target_logits), _logits(draft_logits)
    code = load().tt_verify(ctypes.byref(batch._c()), _ptr(q_hat), ctypes.byref(Lt),
                            ctypes.byref(Ld) if Ld is not None else None, _ptr(map),
                            ctypes.byref(params._c(keep)), _ptr(ws), ws.numel(),
                            _ptr(o["accepted"]), _ptr(o["next_token"]), _ptr(o["p_hat"]),
                            _ptr(o["lse"]), _ptr(o["status"]), _stream(stream))
    _check("tt_verify", code)
    return o


def _shards(shards):
    """ctypes view of a list of per-shard logits tensors (columns in order)."""
    S = len(shards)
    arr = (_Logits * max(S, 1))()
    col0 = (c_i32 * max(S, 1))()
    c = 0
    for k, t in enumerate(shards):
        arr[k] = _logits(t)
        col0[k] = c
        c += t.shape[1]
    return _Shards(S, arr, col0), (arr, col0)


def sharded_workspace(batch: Batch, shards, device="cuda") -> torch.Tensor:
    """Scratch for tt_verify_sharded with these shards."""
    sh, keep = _shards(shards)
    n = int(load().tt_sharded_workspace_bytes(ctypes.byref(batch._c()), ctypes.byref(sh)))
    if n == 0:
        raise TTError("tt_sharded_workspace_bytes", TT_ERR_INVALID_ARG, "invalid argument")
    return torch.empty(n, dtype=torch.uint8, device=device)


def tt_verify_sharded(batch: Batch, q_hat: torch.Tensor, shards, params: Params, *,
                      ws=None, out=None, stream=None, summaries: bool = False) -> dict:
    """Verification over target rows split by columns into len(shards) logits
    tensors (shard k holds the next shards[k].shape[1] columns), emulating a
    vocabulary-sharded target on one GPU; results as tt_verify's, next_token a
    column of the whole row. summaries=True also returns the gathered per-shard
    records [S, n_target + B, 4] (max, sum hi, sum lo, scored logit or NaN)."""
    dev = batch.target_off.device
    o = dict(out or {})
    o.setdefault("accepted", _empty(batch.B, torch.int32, dev))
    o.setdefault("next_token", _empty(batch.B, torch.int32, dev))
    o.setdefault("status", _empty(batch.B, torch.int32, dev))
    o.setdefault("p_hat", _empty(batch.n_target, torch.float32, dev))
    o.setdefault("lse", _empty(batch.n_target + batch.B, torch.float32, dev))
    rows = batch.n_target + batch.B
    if summaries:
        o.setdefault("summaries", torch.empty((len(shards), rows, 4), dtype=torch.float32,
                                              device=dev))
    sh, keep_sh = _shards(shards)
    L = load()
    if ws is None:
        ws = sharded_workspace(batch, shards, dev)
    keep = []
    code = L.tt_verify_sharded(ctypes.byref(batch._c()), _ptr(q_hat), ctypes.byref(sh),
                               ctypes.byref(params._c(keep)), _ptr(ws), ws.numel(),
                               _ptr(o["accepted"]), _ptr(o["next_token"]), _ptr(o["p_hat"]),
                               _ptr(o["lse"]), _ptr(o.get("summaries")), _ptr(o["status"]),
                               _stream(stream))
    _check("tt_verify_sharded", code)
    return o


STEP_OUTPUTS = ("accepted", "next_token", "status", "path", "path_len", "cost", "map", "q_hat",
                "p_hat", "lse")


def step_outputs(batch: Batch, device="cuda", full: bool = True) -> dict:
    """Output tensors of tt_step (the optional ones only when ``full``)."""
    o = {"accepted": _empty(batch.B, torch.int32, device),
         "next_token": _empty(batch.B, torch.int32, device),
         "status": _empty(batch.B, torch.int32, device)}
    if full:
        o["path"] = _empty(2 * (batch.n_draft + batch.n_target), torch.int32, device)
        o["path_len"] = _empty(batch.B, torch.int32, device)
        o["cost"] = _empty(batch.B, torch.int32, device)
        o["map"] = _empty(batch.n_target, torch.int32, device)
        o["q_hat"] = _empty(batch.n_target, torch.float32, device)
        o["p_hat"] = _empty(batch.n_target, torch.float32, device)
        o["lse"] = _empty(batch.n_target + batch.B, torch.float32, device)
    return o


class StepCall:
    """A prepared tt_step call: the ctypes argument blocks are built once, so a
    step costs one foreign call (used by the benchmark's timed loop)."""

    def __init__(self, batch: Batch, vd: VocabTable, vt: VocabTable, draft_logits, target_logits,
                 params: Params, *, draft_probs=None, ws=None, out=None, stream=None):
        dev = batch.target_off.device
        self.out = out if out is not None else step_outputs(batch, dev)
        if ws is None:
            Vd = draft_logits.shape[1] if draft_logits is not None else 0
            ws = workspace(batch, Vd, target_logits.shape[1], dev, params)
        self._keep = [batch, vd, vt, draft_logits, target_logits, draft_probs, ws, self.out]
        self._b = batch._c()
        self._vd = vd._c()
        self._vt = vt._c()
        self._ld = _logits(draft_logits)
        self._lt = _logits(target_logits)
        self._prm = params._c(self._keep)
        self._ws = ws
        o = self.out
        self._out = _StepOut(*[_ptr(o.get(k)) for k in STEP_OUTPUTS])
        self._probs = _ptr(draft_probs)
        self._stream = _stream(stream)
        self._lib = load()
        self._ev = (c_p * 4)()
        self._ev_ptr = ctypes.cast(self._ev, c_p)

    def __call__(self, events=None) -> dict:
        """One step; ``events`` (4 raw cudaEvent_t handles) are recorded around
        the align, row-pass and decision kernels when given."""
        if events is not None:
            for i in range(4):
                self._ev[i] = events[i]
            self._prm.events = self._ev_ptr
        else:
            self._prm.events = None
        code = self._lib.tt_step(ctypes.byref(self._b), ctypes.byref(self._vd),
                                 ctypes.byref(self._vt),
                                 ctypes.byref(self._ld) if self._ld is not None else None,
                                 self._probs, ctypes.byref(self._lt), ctypes.byref(self._prm),
                                 _ptr(self._ws), self._ws.numel(), ctypes.byref(self._out),
                                 self._stream)
        _check("tt_step", code)
        return self.out


def tt_step(batch: Batch, vd: VocabTable, vt: VocabTable, draft_logits, target_logits,
            params: Params, *, draft_probs=None, ws=None, out=None, stream=None) -> dict:
    return StepCall(batch, vd, vt, draft_logits, target_logits, params, draft_probs=draft_probs,
                    ws=ws, out=out, stream=stream)()


def tt_step_noalloc(batch: Batch, vd: VocabTable, vt: VocabTable, draft_logits, target_logits,
                    params: Params, *, draft_probs=None, out=None, stream=None) -> dict:
    """tt_step without a workspace, for callers that cannot allocate device
    memory: the library's own fixed scratch (TT_NOALLOC_SCRATCH_BYTES per GPU)
    is used instead. Outputs are the caller's (allocated here only when not
    given). Calls that overlap on the GPU share that scratch and must be ordered."""
    dev = batch.target_off.device
    o = out if out is not None else step_outputs(batch, dev)
    keep = []
    Ld, Lt = _logits(draft_logits), _logits(target_logits)
    so = _StepOut(*[_ptr(o.get(k)) for k in STEP_OUTPUTS])
    code = load().tt_step_noalloc(ctypes.byref(batch._c()), ctypes.byref(vd._c()),
                                  ctypes.byref(vt._c()),
                                  ctypes.byref(Ld) if Ld is not None else None,
                                  _ptr(draft_probs), ctypes.byref(Lt),
                                  ctypes.byref(params._c(keep)), ctypes.byref(so),
                                  _stream(stream))
    _check("tt_step_noalloc", code)
    return o


def tt_status_string(code: int) -> str:
    return load().tt_status_string(int(code)).decode()


def tt_version() -> int:
    return int(load().tt_version())


# ------------------------------------------------------------- workloads

def device_inputs(wl, device="cuda") -> dict:
    """Moves a synthetic workload (see ``workload``) to the device as binding
    arguments: batch, vocab tables and logits."""
    batch = Batch.from_host(wl.draft_off, wl.draft_ids, wl.target_off, wl.target_ids,
                            wl.draft_cols, wl.target_cols, device=device)
    if getattr(wl, "hist_off_d", None) is not None or getattr(wl, "hist_off_t", None) is not None:
        batch = batch.with_history(wl.hist_off_d, wl.hist_cols_d, wl.hist_off_t, wl.hist_cols_t)
    return dict(batch=batch, vd=VocabTable.from_host(wl.vd.blob, wl.vd.off, device),
                vt=VocabTable.from_host(wl.vt.blob, wl.vt.off, device),
                draft_logits=wl.draft_logits.to(device), target_logits=wl.target_logits.to(device),
                params=Params(window=wl.spec.window, temp_draft=wl.spec.temp_draft,
                              temp_target=wl.spec.temp_target, seed=wl.spec.seed))


# ------------------------------------------------ re-encoding and its checks

def vocab_index(blob, offsets, device="cuda") -> torch.Tensor:
    """Re-encoding index of a target vocabulary (tt_vocab_index_build on host
    arrays), copied to the device once; pass it to tt_encode."""
    import numpy as np
    blob = np.ascontiguousarray(np.asarray(blob, dtype=np.uint8))
    offsets = np.ascontiguousarray(np.asarray(offsets, dtype=np.int64))
    n_tokens = len(offsets) - 1
    L = load()
    nbytes = int(L.tt_vocab_index_bytes(n_tokens, int(offsets[-1]) if n_tokens > 0 else 0))
    host = np.zeros(nbytes, np.uint8)
    code = L.tt_vocab_index_build(blob.ctypes.data if blob.size else None, offsets.ctypes.data,
                                  n_tokens, host.ctypes.data, nbytes)
    _check("tt_vocab_index_build", code)
    return torch.from_numpy(host).to(device)


def tt_encode_workspace_bytes(B: int, max_m: int) -> int:
    return int(load().tt_encode_workspace_bytes(int(B), int(max_m)))


def tt_encode(draft_off: torch.Tensor, draft_ids: torch.Tensor, vd: VocabTable, vt: VocabTable,
              vt_index: torch.Tensor, max_m: int, *, capacity: Optional[int] = None, out=None,
              ws=None, stream=None) -> dict:
    """T_b = encode_t(decode_d(D_b)) on the device; returns target_off, target_ids
    (capacity long) and status."""
    dev = draft_off.device
    B = draft_off.numel() - 1
    n_draft = draft_ids.numel()
    if capacity is None:
        capacity = B * int(max_m)
    o = dict(out or {})
    o.setdefault("target_off", _empty(B + 1, torch.int32, dev))
    o.setdefault("target_ids", _empty(capacity, torch.int32, dev))
    o.setdefault("status", _empty(B, torch.int32, dev))
    if ws is None:
        ws = torch.empty(max(tt_encode_workspace_bytes(B, max_m), 256), dtype=torch.uint8,
                         device=dev)
    code = load().tt_encode(B, n_draft, _ptr(draft_off), _ptr(draft_ids), ctypes.byref(vd._c()),
                            ctypes.byref(vt._c()), _ptr(vt_index), int(max_m), int(capacity),
                            _ptr(o["target_off"]), _ptr(o["target_ids"]), _ptr(o["status"]),
                            _ptr(ws), ws.numel(), _stream(stream))
    _check("tt_encode", code)
    return o


def tt_consistency(batch: Batch, vd: VocabTable, vt: VocabTable, *, status=None,
                   stream=None) -> torch.Tensor:
    """Lemma-1 byte check of (D, T) per request."""
    st = status if status is not None else _empty(batch.B, torch.int32, batch.draft_off.device)
    code = load().tt_consistency(ctypes.byref(batch._c()), ctypes.byref(vd._c()),
                                 ctypes.byref(vt._c()), _ptr(st), _stream(stream))
    _check("tt_consistency", code)
    return st


def tt_dpos_hist(batch: Batch, path: torch.Tensor, path_len: torch.Tensor,
                 map: Optional[torch.Tensor], mode: int, n_bins: int, *,
                 hist: Optional[torch.Tensor] = None, stream=None) -> torch.Tensor:
    """Delta-pos histogram of the alignment paths (mode 0) or the map (mode 1),
    added to `hist` (a zeroed int64 tensor is made when none is given)."""
    dev = batch.draft_off.device
    h = hist if hist is not None else torch.zeros(int(n_bins), dtype=torch.int64, device=dev)
    code = load().tt_dpos_hist(ctypes.byref(batch._c()), _ptr(path), _ptr(path_len), _ptr(map),
                               int(mode), int(n_bins), _ptr(h), _stream(stream))
    _check("tt_dpos_hist", code)
    return h
