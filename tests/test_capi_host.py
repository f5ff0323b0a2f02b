"""C ABI tests that need no GPU: the library loads, exports every declared entry
point, and rejects bad descriptions with the right status before any launch."""
import ctypes
import os
import re

import numpy as np
import pytest

from paper_2608_05780_gb300 import _binding as B
from paper_2608_05780_gb300.build import build

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def lib():
    build()
    return B.load()


def _declared_functions():
    names = []
    for h in os.listdir(os.path.join(ROOT, "include")):
        if h.endswith(".h"):
            text = open(os.path.join(ROOT, "include", h)).read()
            text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
            names += re.findall(r"^[A-Za-z_][\w\s\*]*?\b(evisel_\w+)\s*\(", text, flags=re.M)
    return sorted(set(names))


def test_exports_every_declared_symbol(lib):
    declared = _declared_functions()
    assert {"evisel_probe_attention", "evisel_evidence_reduce", "evisel_free"} <= set(declared)
    for name in declared:
        assert hasattr(lib, name), name


def test_strerror(lib):
    for code in range(0, -9, -1):
        assert lib.evisel_strerror(code)
    assert lib.evisel_strerror(-1) == b"invalid argument"


FAKE = 0x7F0000000000   # never dereferenced: validation fails before any device access


def _args(**over):
    p = dict(cu=[0, 300], n_vis=[256], npf=16, hq=4, hkv=2, d=64, tile=64,
             row_ptr=[0, 1, 3, 5, 7], col_idx=[0, 0, 1, 1, 2, 2, 3], q=FAKE, k=FAKE, v=FAKE, o=FAKE, lse=FAKE,
             scale=0.0)
    p.update(over)
    keep = []

    def arr(x):
        a = np.ascontiguousarray(np.asarray(x, dtype=np.int32))
        keep.append(a)
        return a.ctypes.data_as(ctypes.POINTER(ctypes.c_int32))
    a = B.ProbeArgs()
    a.num_videos = len(p["n_vis"])
    a.cu_seqlens_h = arr(p["cu"])
    a.n_vis_h = arr(p["n_vis"])
    a.tokens_per_frame = p["npf"]
    a.hq, a.hkv, a.head_dim, a.tile = p["hq"], p["hkv"], p["d"], p["tile"]
    a.softmax_scale = p["scale"]
    a.q, a.k, a.v, a.o, a.lse = p["q"], p["k"], p["v"], p["o"], p["lse"]
    a.mask_row_ptr_h = arr(p["row_ptr"])
    a.mask_col_idx_h = arr(p["col_idx"] or [0])
    a.cross_frame = p.get("cross_frame", 0)
    return a, keep


@pytest.mark.parametrize("over,code", [
    (dict(d=96), -2),
    (dict(d=32), -2),
    (dict(tile=32), -2),
    (dict(hq=5, hkv=2), -2),
    (dict(npf=3), -2),
    (dict(npf=128), -2),
    (dict(npf=2), -2),
    (dict(hq=0), -1),
    (dict(q=0), -1),
    (dict(lse=0), -1),
    (dict(o=FAKE + 8), -1),
    (dict(n_vis=[250]), -1),
    (dict(n_vis=[320]), -1),
    (dict(cu=[0, -5], n_vis=[0]), -1),
    (dict(cu=[1, 300]), -1),
    (dict(scale=float("nan")), -1),
    (dict(scale=-1.0), -1),
    (dict(col_idx=[0, 1, 0, 1, 2, 2, 3]), -3),       # row 1 lacks its diagonal
    (dict(col_idx=[0, 0, 1, 2, 1, 2, 3]), -3),       # row 2 not ascending
    (dict(col_idx=[0, 0, 1, 1, 2, 2, 4]), -3),       # non-causal tile
    (dict(col_idx=[0, 0, 1, -1, 2, 2, 3]), -3),      # negative tile
    (dict(row_ptr=[0, 1, 1, 5, 7]), -3),             # empty row
    (dict(row_ptr=[1, 1, 3, 5, 7]), -3),
    (dict(cross_frame=2), -1),
    (dict(cross_frame=1, npf=8, n_vis=[256]), -2),   # cross-frame partials need N_v >= 16
])
def test_validation_rejects(lib, over, code):
    a, keep = _args(**over)
    ws = ctypes.c_void_p(None)
    rc = lib.evisel_probe_attention(ctypes.byref(a), None, ctypes.byref(ws))
    assert rc == code, lib.evisel_last_error()
    assert ws.value is None          # nothing allocated, nothing launched
    assert lib.evisel_last_error()


def test_null_workspace_pointer(lib):
    a, keep = _args()
    assert lib.evisel_probe_attention(ctypes.byref(a), None, None) == -1


def test_evidence_without_probe(lib):
    assert lib.evisel_evidence_reduce(None, None, None, None, None, 0, None) == -1


def test_cross_frame_without_workspace(lib):
    a, keep = _args(cross_frame=1)
    assert lib.evisel_cross_frame_evidence(ctypes.byref(a), None, None, None, 0, None) == -1


def test_noalloc_rejects_cross_frame(lib):
    a, keep = _args(cross_frame=1)
    st = ctypes.c_int(0)
    rc = lib.evisel_probe_evidence_noalloc(ctypes.byref(a), ctypes.c_void_p(FAKE), ctypes.c_void_p(FAKE),
                                           ctypes.c_void_p(FAKE), ctypes.c_void_p(FAKE), 0, None, ctypes.byref(st))
    assert rc == -2, lib.evisel_last_error()


def test_free_null_is_safe(lib):
    lib.evisel_free(None)
    assert lib.evisel_workspace_bytes(None) == 0


def test_binding_fails_loudly_without_library(tmp_path):
    saved = B._lib
    B._lib = None
    try:
        with pytest.raises(RuntimeError, match="not built"):
            B.load(str(tmp_path / "missing.so"))
    finally:
        B._lib = saved


@pytest.mark.parametrize("block,tau,over,code", [
    (24, 0.97, {}, -2),                  # block not a power of two
    (8, 0.97, {}, -2),                   # block below 16
    (32, 0.97, {}, -2),                  # block above N_v (16): it must divide the frames
    (16, 0.0, {}, -1),                   # tau_p outside (0, 1]
    (16, 1.5, {}, -1),
    (16, float("nan"), {}, -1),
    (16, 0.97, dict(q=FAKE + 8), -1),    # q not 16-byte aligned (TMA)
    (16, 0.97, dict(d=96), -2),
    (16, 0.97, dict(hq=5, hkv=2), -2),
    (16, 0.97, dict(n_vis=[250]), -1),   # n_vis not a multiple of N_v
    (16, 0.97, dict(scale=-1.0), -1),
])
def test_topp_validation_rejects(lib, block, tau, over, code):
    a, keep = _args(**over)
    ws = ctypes.c_void_p(None)
    rc = lib.evisel_topp_mask(ctypes.byref(a), block, tau, ctypes.c_void_p(FAKE), None, None, ctypes.byref(ws))
    assert rc == code, lib.evisel_last_error()
    assert ws.value is None          # nothing allocated, nothing launched
    assert lib.evisel_last_error()


def test_topp_null_keep_and_workspace_pointer(lib):
    a, keep = _args()
    ws = ctypes.c_void_p(None)
    assert lib.evisel_topp_mask(ctypes.byref(a), 16, 0.97, None, None, None, ctypes.byref(ws)) == -1
    assert lib.evisel_topp_mask(ctypes.byref(a), 16, 0.97, ctypes.c_void_p(FAKE), None, None, None) == -1


def test_coarse_evidence_without_workspace(lib):
    a, keep = _args()
    fake = ctypes.c_void_p(FAKE)
    assert lib.evisel_coarse_evidence(ctypes.byref(a), None, 16, fake, fake, fake, fake, fake, 0, None) == -1
