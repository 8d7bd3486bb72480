"""The C-ABI library builds for sm_103a, loads without a GPU, exports every
entry point include/tt.h declares, and rejects bad arguments on the host
before anything reaches the GPU (no compute call is made here)."""
import ctypes
import os
import re

import pytest
import torch

import paper_2510_15545_gb300 as tt
from paper_2510_15545_gb300 import _build, binding

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "tt.h")


@pytest.fixture(scope="module")
def lib():
    _build.build()
    return tt.load()


def declared_functions():
    src = open(HEADER).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    return sorted(set(re.findall(r"^\s*(?:const\s+)?[\w ]+?\**\s*\b(tt_\w+)\s*\(", src, flags=re.M)))


def test_every_declared_symbol_is_exported(lib):
    names = declared_functions()
    assert {"tt_align", "tt_transfer", "tt_verify", "tt_step", "tt_workspace_bytes",
            "tt_status_string"} <= set(names)
    for n in names:
        assert hasattr(lib, n), n
    assert set(binding.EXPORTS) == set(names)


def test_library_is_built_for_sm103a():
    objs = [os.path.join(_build.OUT_DIR, s.replace(".cu", ".o")) for s in _build.SOURCES]
    assert all(os.path.exists(o) for o in objs)
    assert "arch=compute_103a,code=sm_103a" in " ".join(_build.ARCH)


def test_struct_layouts_match_the_header():
    # sizes/offsets of the C structs under the LP64 ABI (x86-64 and aarch64 alike)
    assert ctypes.sizeof(binding._Params) == 64
    assert binding._Params.seed.offset == 16 and binding._Params.events.offset == 32
    assert binding._Params.top_k_draft.offset == 40 and binding._Params.top_p_target.offset == 52
    assert binding._Params.rep_penalty_target.offset == 60
    assert ctypes.sizeof(binding._Logits) == 32 and binding._Logits.row_stride.offset == 16
    assert ctypes.sizeof(binding._Vocab) == 32 and binding._Vocab.n_bytes.offset == 24
    assert binding._Batch.draft_off.offset == 24 and binding._Batch.hist_off_d.offset == 72
    assert binding._Batch.n_hist_t.offset == 108 and ctypes.sizeof(binding._Batch) == 112
    assert ctypes.sizeof(binding._StepOut) == 80
    assert ctypes.sizeof(binding._Shards) == 24 and binding._Shards.col0.offset == 16


def test_status_strings_and_version(lib):
    assert tt.tt_status_string(0) == "ok"
    assert tt.tt_status_string(1) == "invalid argument"
    assert tt.tt_status_string(2) == "unsupported configuration"
    assert tt.tt_version() >= 100


def _batch_host():
    # pointers are never dereferenced: every call below fails validation first
    return tt.Batch.from_host([0, 2], [1, 2], [0, 3], [1, 2, 3], device="cpu")


def test_host_validation_rejects_bad_arguments(lib):
    b = _batch_host()
    vd = tt.VocabTable.from_host([97, 98, 99], [0, 1, 2, 3], device="cpu")
    prm = binding.Params()
    keep = []
    P = ctypes.byref
    # B < 0
    bad = b._c()
    bad.B = -1
    assert lib.tt_align(P(bad), P(vd._c()), P(vd._c()), P(prm._c(keep)), None, None, None, None,
                        None, None) == binding.TT_ERR_INVALID_ARG
    # max_k above the cap
    bad = b._c()
    bad.max_k = 300
    assert lib.tt_align(P(bad), P(vd._c()), P(vd._c()), P(prm._c(keep)), None, None, None, None,
                        ctypes.c_void_p(16), None) == binding.TT_ERR_INVALID_ARG
    # non-positive temperature
    p2 = binding.Params(temp_target=0.0)._c(keep)
    assert lib.tt_align(P(b._c()), P(vd._c()), P(vd._c()), P(p2), None, None, None, None,
                        ctypes.c_void_p(16), None) == binding.TT_ERR_INVALID_ARG
    # missing status output
    assert lib.tt_align(P(b._c()), P(vd._c()), P(vd._c()), P(prm._c(keep)), None, None, None,
                        None, None, None) == binding.TT_ERR_INVALID_ARG
    # misaligned logits rows
    lg = binding._Logits(16 + 4, binding.TT_F32, 100, 100, 10)
    out = binding._StepOut(16, 16, 16, None, None, None, None, None, None, None)
    assert lib.tt_step(P(b._c()), P(vd._c()), P(vd._c()), P(lg), None, P(lg), P(prm._c(keep)),
                       ctypes.c_void_p(256), 1 << 30, P(out), None) == binding.TT_ERR_INVALID_ARG
    # row stride not a multiple of 16 bytes
    lg = binding._Logits(256, binding.TT_F32, 101, 101, 10)
    assert lib.tt_step(P(b._c()), P(vd._c()), P(vd._c()), P(lg), None, P(lg), P(prm._c(keep)),
                       ctypes.c_void_p(256), 1 << 30, P(out), None) == binding.TT_ERR_INVALID_ARG
    # workspace too small
    lg = binding._Logits(256, binding.TT_F32, 128, 128, 10)
    assert lib.tt_step(P(b._c()), P(vd._c()), P(vd._c()), P(lg), None, P(lg), P(prm._c(keep)),
                       ctypes.c_void_p(256), 8, P(out), None) == binding.TT_ERR_INVALID_ARG
    # full_q needs draft and target rows of one width
    lg2 = binding._Logits(256, binding.TT_F32, 64, 64, 10)
    pq = binding.Params(full_q=True)._c(keep)
    assert lib.tt_step(P(b._c()), P(vd._c()), P(vd._c()), P(lg2), None, P(lg), P(pq),
                       ctypes.c_void_p(256), 1 << 30, P(out), None) == binding.TT_ERR_INVALID_ARG
    # an empty batch is a no-op for every entry point (nothing is launched,
    # no output or workspace is needed)
    e = tt.Batch.from_host([0], [], [0], [], device="cpu")
    assert lib.tt_align(P(e._c()), P(vd._c()), P(vd._c()), P(prm._c(keep)), None, None, None,
                        None, None, None) == binding.TT_OK
    assert lib.tt_transfer(P(e._c()), None, P(lg), None, P(prm._c(keep)), None, 0, None, None,
                           None) == binding.TT_OK
    assert lib.tt_verify(P(e._c()), None, P(lg), None, None, P(prm._c(keep)), None, 0, None,
                         None, None, None, None, None) == binding.TT_OK
    assert lib.tt_step(P(e._c()), P(vd._c()), P(vd._c()), P(lg), None, P(lg), P(prm._c(keep)),
                       None, 0, P(out), None) == binding.TT_OK
    sh, _k = _shards([64, 64])
    assert lib.tt_verify_sharded(P(e._c()), None, P(sh), P(prm._c(keep)), None, 0, None, None,
                                 None, None, None, None, None) == binding.TT_OK


def _shards(widths, col0=None):
    arr = (binding._Logits * len(widths))()
    c0 = (ctypes.c_int32 * len(widths))()
    c = 0
    for k, w in enumerate(widths):
        arr[k] = binding._Logits(256 * (k + 1), binding.TT_F32, w, (w + 3) // 4 * 4, 10)
        c0[k] = c if col0 is None else col0[k]
        c += w
    return binding._Shards(len(widths), arr, c0), (arr, c0)


def test_sharded_verify_host_rules(lib):
    b = _batch_host()
    keep = []
    P = ctypes.byref
    prm = binding.Params()._c(keep)
    one = lib.tt_sharded_workspace_bytes(P(b._c()), P(_shards([100])[0]))
    three = lib.tt_sharded_workspace_bytes(P(b._c()), P(_shards([40, 4096, 3000])[0]))
    assert 0 < one < three
    # shards must tile the row from column 0, in order, and number 1..8
    for sh, _ in (_shards([40, 60], col0=[0, 41]), _shards([40, 60], col0=[1, 41]),
                  _shards([8] * (binding.TT_MAX_SHARDS + 1))):
        assert lib.tt_sharded_workspace_bytes(P(b._c()), P(sh)) == 0
        assert lib.tt_verify_sharded(P(b._c()), ctypes.c_void_p(16), P(sh), P(prm),
                                     ctypes.c_void_p(256), 1 << 30, ctypes.c_void_p(16),
                                     ctypes.c_void_p(16), None, None, None, ctypes.c_void_p(16),
                                     None) == binding.TT_ERR_INVALID_ARG
    sh, _ = _shards([40, 60])
    call = lambda p, n=1 << 30: lib.tt_verify_sharded(
        P(b._c()), ctypes.c_void_p(16), P(sh), P(p), ctypes.c_void_p(256), n, ctypes.c_void_p(16),
        ctypes.c_void_p(16), None, None, None, ctypes.c_void_p(16), None)
    # one-hot transfer without filters only
    assert call(binding.Params(full_q=True)._c(keep)) == binding.TT_ERR_UNSUPPORTED
    assert call(binding.Params(top_k_target=5)._c(keep)) == binding.TT_ERR_UNSUPPORTED
    # workspace too small
    assert call(prm, 8) == binding.TT_ERR_INVALID_ARG


def test_workspace_bytes_grow_with_the_batch(lib):
    small = tt.Batch.from_host([0, 2], [1, 2], [0, 3], [1, 2, 3], device="cpu")
    big = tt.Batch.from_host([0, 20], list(range(20)), [0, 30], list(range(30)), device="cpu")
    assert tt.tt_workspace_bytes(big, 32000, 151936) > tt.tt_workspace_bytes(small, 32000, 151936)
    assert tt.tt_workspace_bytes(small, 32000, 151936) % 256 == 0


def test_binding_fails_loudly_without_the_library(monkeypatch, tmp_path):
    monkeypatch.setattr(binding, "_lib", None)
    monkeypatch.setattr(binding, "lib_path", lambda: str(tmp_path / "missing.so"))
    with pytest.raises(RuntimeError, match="not built"):
        binding.load()


def test_workspace_of_filter_families(lib):
    """Host sizing of the workspace with sampling filters: top-k families add
    their per-unit lists (k rounded up to even entries of 8 bytes per 8 KB
    unit) and kept sets; nucleus families (top-p without top-k) add only a
    float per 2048-column chunk and a header per row, no lists."""
    b = tt.Batch.from_host([0, 8], list(range(8)), [0, 10], list(range(10)), device="cpu")
    V = 151936
    plain = tt.tt_workspace_bytes(b, V, V, tt.Params())
    topk = tt.tt_workspace_bytes(b, V, V, tt.Params(top_k_draft=20, top_k_target=20))
    nuc = tt.tt_workspace_bytes(b, V, V, tt.Params(top_p_draft=0.9, top_p_target=0.9))
    units = (V + 2047) // 2048  # fp32 sizing: 2048 columns per unit
    rows = 8 + 10 + 1           # draft rows, target rows (with the bonus row)
    lists = rows * units * 20 * 8
    assert topk - plain >= lists
    assert plain < nuc < plain + rows * (units * 4 + 64) + 8 * 256
    assert nuc < topk
