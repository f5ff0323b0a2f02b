"""ctypes binding of libevisel.so: argument marshalling only.

The functions carry the C ABI's names (include/evisel.h). PyTorch provides
device memory and the current CUDA stream; every step of the probe runs in the
library's sm_103a kernels. There is no CPU fallback: if the library cannot be
loaded the calls raise.
"""
from __future__ import annotations

import ctypes
import os

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "libevisel.so")

EVISEL_OK = 0
_ERRORS = {-1: "EINVAL", -2: "EUNSUPPORTED", -3: "EMASK", -4: "ECUDA", -5: "ENOMEM", -6: "ETIMEOUT",
           -7: "EBOUNDS", -8: "ESTATE"}


class EviselError(RuntimeError):
    def __init__(self, code, msg):
        super().__init__(f"{_ERRORS.get(code, code)} ({code}): {msg}")
        self.code = code


class ProbeArgs(ctypes.Structure):
    _fields_ = [
        ("num_videos", ctypes.c_int32),
        ("cu_seqlens_h", ctypes.POINTER(ctypes.c_int32)),
        ("n_vis_h", ctypes.POINTER(ctypes.c_int32)),
        ("tokens_per_frame", ctypes.c_int32),
        ("hq", ctypes.c_int32),
        ("hkv", ctypes.c_int32),
        ("head_dim", ctypes.c_int32),
        ("tile", ctypes.c_int32),
        ("softmax_scale", ctypes.c_float),
        ("q", ctypes.c_void_p),
        ("k", ctypes.c_void_p),
        ("v", ctypes.c_void_p),
        ("mask_row_ptr_h", ctypes.POINTER(ctypes.c_int32)),
        ("mask_col_idx_h", ctypes.POINTER(ctypes.c_int32)),
        ("o", ctypes.c_void_p),
        ("lse", ctypes.c_void_p),
        ("cross_frame", ctypes.c_int32),
        ("text_evidence", ctypes.c_int32),
        ("keep", ctypes.c_void_p),
        ("keep_words", ctypes.c_int32),
        ("keep_block", ctypes.c_int32),
    ]


EXPORTS = ["evisel_probe_attention", "evisel_evidence_reduce", "evisel_free", "evisel_status",
           "evisel_strerror", "evisel_last_error", "evisel_workspace_bytes", "evisel_build_id"]

_lib = None


def load(path: str = LIB_PATH):
    """Loads the library (once) and declares the C signatures."""
    global _lib
    if _lib is not None:
        return _lib
    if not os.path.exists(path):
        raise RuntimeError(f"libevisel.so is not built ({path}); run paper_2608_05780_gb300.build.build()")
    lib = ctypes.CDLL(path)
    vp, i32 = ctypes.c_void_p, ctypes.c_int
    lib.evisel_probe_attention.argtypes = [ctypes.POINTER(ProbeArgs), vp, ctypes.POINTER(vp)]
    lib.evisel_probe_attention.restype = i32
    lib.evisel_evidence_reduce.argtypes = [vp, vp, vp, vp, vp, i32, vp]
    lib.evisel_evidence_reduce.restype = i32
    lib.evisel_free.argtypes = [vp]
    lib.evisel_free.restype = None
    lib.evisel_status.argtypes = [vp]
    lib.evisel_status.restype = i32
    lib.evisel_strerror.argtypes = [i32]
    lib.evisel_strerror.restype = ctypes.c_char_p
    lib.evisel_last_error.argtypes = []
    lib.evisel_last_error.restype = ctypes.c_char_p
    lib.evisel_workspace_bytes.argtypes = [vp]
    lib.evisel_workspace_bytes.restype = ctypes.c_int64
    lib.evisel_build_id.argtypes = []
    lib.evisel_build_id.restype = ctypes.c_char_p
    lib.evisel_probe_evidence_noalloc.argtypes = [ctypes.POINTER(ProbeArgs), vp, vp, vp, vp, i32, vp,
                                                  ctypes.POINTER(ctypes.c_int)]
    lib.evisel_probe_evidence_noalloc.restype = i32
    lib.evisel_intra_frame_evidence.argtypes = [ctypes.POINTER(ProbeArgs), vp, vp, i32, vp]
    lib.evisel_intra_frame_evidence.restype = i32
    lib.evisel_cross_frame_evidence.argtypes = [ctypes.POINTER(ProbeArgs), vp, vp, vp, i32, vp]
    lib.evisel_cross_frame_evidence.restype = i32
    lib.evisel_topp_mask.argtypes = [ctypes.POINTER(ProbeArgs), i32, ctypes.c_float, vp, vp, vp, ctypes.POINTER(vp)]
    lib.evisel_topp_mask.restype = i32
    lib.evisel_coarse_evidence.argtypes = [ctypes.POINTER(ProbeArgs), vp, i32, vp, vp, vp, vp, vp, i32, vp]
    lib.evisel_coarse_evidence.restype = i32
    lib.evisel_selftest_wait.argtypes = [i32, i32, vp, ctypes.POINTER(ctypes.c_int)]
    lib.evisel_selftest_wait.restype = i32
    _lib = lib
    return lib


def _check(rc):
    if rc != EVISEL_OK:
        raise EviselError(rc, _lib.evisel_last_error().decode())


def _i32(a):
    arr = np.ascontiguousarray(np.asarray(a, dtype=np.int32))
    return arr, arr.ctypes.data_as(ctypes.POINTER(ctypes.c_int32))


def _stream_handle(stream):
    import torch
    s = torch.cuda.current_stream() if stream is None else stream
    return ctypes.c_void_p(s.cuda_stream)


class Workspace:
    """Owner of an evisel_ws* (freed with evisel_free)."""

    def __init__(self):
        self.ptr = ctypes.c_void_p(None)

    @property
    def nbytes(self):
        return int(load().evisel_workspace_bytes(self.ptr))

    def free(self):
        if self.ptr.value:
            load().evisel_free(self.ptr)
            self.ptr = ctypes.c_void_p(None)

    def __del__(self):
        try:
            self.free()
        except Exception:
            pass


def make_args(q, k, v, cu_seqlens, n_vis, tokens_per_frame, tile, row_ptr, col_idx, o, lse,
              softmax_scale=0.0, cross_frame=False, text_evidence=False, keep=None, keep_block=0):
    """Fills the C struct; returns (struct, keepalive) - keepalive holds the host arrays."""
    cu, cu_p = _i32(cu_seqlens)
    nv, nv_p = _i32(n_vis)
    rp, rp_p = _i32(row_ptr)
    ci, ci_p = _i32(col_idx if len(col_idx) else np.zeros(1, np.int32))
    a = ProbeArgs()
    a.num_videos = len(nv)
    a.cu_seqlens_h = cu_p
    a.n_vis_h = nv_p
    a.tokens_per_frame = int(tokens_per_frame)
    a.hq = int(q.shape[1])
    a.hkv = int(k.shape[1])
    a.head_dim = int(q.shape[2])
    a.tile = int(tile)
    a.softmax_scale = float(softmax_scale)
    a.q, a.k, a.v = q.data_ptr(), k.data_ptr(), v.data_ptr()
    a.mask_row_ptr_h = rp_p
    a.mask_col_idx_h = ci_p
    a.o, a.lse = o.data_ptr(), lse.data_ptr()
    a.cross_frame = int(bool(cross_frame))
    a.text_evidence = int(bool(text_evidence))
    if keep is not None:
        a.keep = keep.data_ptr()
        a.keep_words = int(keep.shape[1])
        a.keep_block = int(keep_block)
    return a, (cu, nv, rp, ci)


def evisel_probe_attention(q, k, v, cu_seqlens, n_vis, tokens_per_frame, tile, row_ptr, col_idx,
                           ws=None, o=None, lse=None, softmax_scale=0.0, stream=None, cross_frame=False,
                           text_evidence=False, keep=None, keep_block=0):
    """Block-sparse GQA varlen probe attention. q/k/v: CUDA bf16 [N, H, d].
    ``cross_frame`` also keeps the partials evisel_cross_frame_evidence reads;
    ``text_evidence`` makes evisel_evidence_reduce recompute the text-row
    probabilities from q and k instead of spilling the logits; ``keep`` (from
    evisel_topp_mask, with its ``keep_block``) restricts every row to its
    retained blocks.

    Returns (o [N, hq, d] bf16, lse [hq, N] fp32, ws).
    """
    import torch
    lib = load()
    for t in (q, k, v):
        if not (t.is_cuda and t.dtype == torch.bfloat16 and t.is_contiguous() and t.dim() == 3):
            raise ValueError("q, k, v must be contiguous CUDA bf16 tensors [N, H, d]")
    n, hq, d = q.shape
    if o is None:
        o = torch.empty((n, hq, d), dtype=torch.bfloat16, device=q.device)
    if lse is None:
        lse = torch.empty((hq, n), dtype=torch.float32, device=q.device)
    if ws is None:
        ws = Workspace()
    args, keep = make_args(q, k, v, cu_seqlens, n_vis, tokens_per_frame, tile, row_ptr, col_idx, o, lse,
                           softmax_scale, cross_frame, text_evidence, keep, keep_block)
    _check(lib.evisel_probe_attention(ctypes.byref(args), _stream_handle(stream), ctypes.byref(ws.ptr)))
    del keep
    return o, lse, ws


def evisel_evidence_reduce(ws, hq, n_vis, tokens_per_frame, num_videos, tok=None, frame=None, head=None,
                           aqf=None, accumulate=False, stream=None, device="cuda"):
    """Token / frame / head / A_qf evidence of the last probe on ``ws``.

    Returns (tok [hq, sum n_vis], frame [hq, sum T], head [B, hq], aqf [sum T]).
    """
    import torch
    lib = load()
    total_vis = int(np.sum(n_vis))
    total_frames = total_vis // int(tokens_per_frame)
    f32 = dict(dtype=torch.float32, device=device)
    if tok is None:
        tok = torch.zeros((hq, total_vis), **f32)
    if frame is None:
        frame = torch.zeros((hq, total_frames), **f32)
    if head is None:
        head = torch.zeros((num_videos, hq), **f32)
    if aqf is None:
        aqf = torch.zeros((total_frames,), **f32)
    _check(lib.evisel_evidence_reduce(ws.ptr, tok.data_ptr(), frame.data_ptr(), head.data_ptr(),
                                      aqf.data_ptr(), int(bool(accumulate)), _stream_handle(stream)))
    return tok, frame, head, aqf


def evisel_status(ws):
    return int(load().evisel_status(ws.ptr))


def evisel_free(ws):
    ws.free()


NOALLOC_SCRATCH_BYTES = 64 << 20


def evisel_probe_evidence_noalloc(q, k, v, cu_seqlens, n_vis, tokens_per_frame, tile, row_ptr, col_idx, o, lse,
                                  tok, frame, head, aqf, accumulate=False, softmax_scale=0.0, stream=None,
                                  wait_status=True, text_evidence=False):
    """Probe + evidence through the entry point that allocates nothing.

    For callers that cannot let the library call cudaMalloc: every output
    (o, lse and the four maps) is passed in, and the library's scratch is a
    fixed 64 MiB static device array (problems that need more are rejected;
    ``text_evidence`` drops the text-row logit spill, the largest part).
    Returns the device status word when ``wait_status`` (the call then waits
    for the stream), else None.
    """
    lib = load()
    args, keep = make_args(q, k, v, cu_seqlens, n_vis, tokens_per_frame, tile, row_ptr, col_idx, o, lse,
                           softmax_scale, text_evidence=text_evidence)
    status = ctypes.c_int(0)
    _check(lib.evisel_probe_evidence_noalloc(ctypes.byref(args), tok.data_ptr(), frame.data_ptr(), head.data_ptr(),
                                             aqf.data_ptr(), int(bool(accumulate)), _stream_handle(stream),
                                             ctypes.byref(status) if wait_status else None))
    del keep
    return int(status.value) if wait_status else None


def evisel_selftest_wait(timeout_us, arrive, stream=None):
    """Runs the kernels' bounded wait on a barrier that is (arrive) or is not
    completed; returns the device status word (0, or EVISEL_ETIMEOUT when the
    wait gave up)."""
    lib = load()
    status = ctypes.c_int(1)
    _check(lib.evisel_selftest_wait(int(timeout_us), int(bool(arrive)), _stream_handle(stream), ctypes.byref(status)))
    return int(status.value)


def evisel_intra_frame_evidence(q, k, v, cu_seqlens, n_vis, tokens_per_frame, tile, row_ptr, col_idx, o, lse, ws,
                                aif=None, accumulate=False, softmax_scale=0.0, stream=None):
    """Intra-frame cue A_if [sum T, N_v, N_v] (fp32) of the probe that ran on ``ws``
    with these arguments (o and lse are that probe's outputs)."""
    import torch
    lib = load()
    n_vis_np = np.asarray(n_vis, dtype=np.int64)
    frames = int(np.sum(n_vis_np // int(tokens_per_frame)))
    if aif is None:
        aif = torch.zeros((frames, int(tokens_per_frame), int(tokens_per_frame)), dtype=torch.float32,
                          device=q.device)
    args, keep = make_args(q, k, v, cu_seqlens, n_vis, tokens_per_frame, tile, row_ptr, col_idx, o, lse,
                           softmax_scale)
    _check(lib.evisel_intra_frame_evidence(ctypes.byref(args), ws.ptr, aif.data_ptr(), int(bool(accumulate)),
                                           _stream_handle(stream)))
    del keep
    return aif


def evisel_cross_frame_evidence(q, k, v, cu_seqlens, n_vis, tokens_per_frame, tile, row_ptr, col_idx, o, lse, ws,
                                aff=None, eff=None, accumulate=False, softmax_scale=0.0, stream=None):
    """Cross-frame cue A_ff (the videos' [(T-1), (T-1)] blocks back to back,
    fp32) and E_ff [sum T] of the probe that ran on ``ws`` with cross_frame=True
    and these arguments (o and lse are that probe's outputs).

    Returns (aff, eff)."""
    import torch
    lib = load()
    npf = int(tokens_per_frame)
    t = np.asarray(n_vis, dtype=np.int64) // npf
    n_aff = int(np.sum(np.maximum(t - 1, 0) ** 2))
    if aff is None:
        aff = torch.empty(n_aff, dtype=torch.float32, device=q.device)
    if eff is None:
        eff = torch.empty(int(np.sum(t)), dtype=torch.float32, device=q.device)
    args, keep = make_args(q, k, v, cu_seqlens, n_vis, tokens_per_frame, tile, row_ptr, col_idx, o, lse,
                           softmax_scale, True)
    _check(lib.evisel_cross_frame_evidence(ctypes.byref(args), ws.ptr, aff.data_ptr() if n_aff else None,
                                           eff.data_ptr() if eff.numel() else None, int(bool(accumulate)),
                                           _stream_handle(stream)))
    del keep
    return aff, eff


def evisel_topp_mask(q, k, cu_seqlens, n_vis, tokens_per_frame, tile, block, tau_p, ws=None, softmax_scale=0.0,
                     stream=None, union=True):
    """Top-p block retention (Appendix Eq. 6-9): returns (keep, tile_union, ws)
    with keep int32 [hq, W, N] (uint32 bit words), tile_union int32
    [visual row tiles, TW] or None."""
    import torch
    lib = load()
    nv = np.asarray(n_vis, dtype=np.int64)
    cu = np.asarray(cu_seqlens, dtype=np.int64)
    n_text = np.diff(cu) - nv
    nb = nv // int(block) + -(-n_text // int(block))
    n, hq = int(q.shape[0]), int(q.shape[1])
    n_words = max(1, -(-int(nb.max() if nb.size else 0) // 32))
    keep = torch.empty((hq, n_words, n), dtype=torch.int32, device=q.device)
    n_vt = -(-nv // int(tile))
    uni = None
    if union:
        uni = torch.empty((int(n_vt.sum()), max(1, -(-int(n_vt.max() if n_vt.size else 0) // 32))),
                          dtype=torch.int32, device=q.device)
    if ws is None:
        ws = Workspace()
    dummy = torch.empty(0, device=q.device)
    args, keepalive = make_args(q, k, k, cu_seqlens, n_vis, tokens_per_frame, tile, [0], [], dummy, dummy,
                                softmax_scale)
    _check(lib.evisel_topp_mask(ctypes.byref(args), int(block), float(tau_p), keep.data_ptr(),
                                uni.data_ptr() if uni is not None and uni.numel() else None,
                                _stream_handle(stream), ctypes.byref(ws.ptr)))
    del keepalive
    return keep, uni, ws


def tile_union_to_csr(tile_union, n_vis, tile):
    """Host CSR (row_ptr, col_idx) of a tile union from evisel_topp_mask."""
    bits = tile_union.cpu().numpy().view(np.uint32)
    row_ptr, cols = [0], []
    r = 0
    for nv in np.asarray(n_vis, dtype=np.int64):
        for _ in range(-(-int(nv) // int(tile))):
            for w, word in enumerate(bits[r]):
                word = int(word)
                while word:
                    low = word & -word
                    cols.append(w * 32 + low.bit_length() - 1)
                    word ^= low
            row_ptr.append(len(cols))
            r += 1
    return np.array(row_ptr, np.int32), np.array(cols, np.int32)


def evisel_coarse_evidence(q, k, cu_seqlens, n_vis, tokens_per_frame, tile, block, keep, ws, tok=None, frame=None,
                           head=None, aqf=None, accumulate=False, softmax_scale=0.0, stream=None):
    """Evidence maps of the coarse token-level map (Appendix Eq. 10-11) on the
    evisel_topp_mask call that ran on ``ws`` (``keep`` its bits).

    Returns (tok [hq, sum n_vis], frame [hq, sum T], head [B, hq], aqf [sum T])."""
    import torch
    lib = load()
    nv = np.asarray(n_vis, dtype=np.int64)
    hq = int(q.shape[1])
    total_vis = int(nv.sum())
    frames = int((nv // int(tokens_per_frame)).sum())
    dev = q.device
    tok = torch.empty((hq, total_vis), device=dev) if tok is None else tok
    frame = torch.empty((hq, frames), device=dev) if frame is None else frame
    head = torch.empty((len(nv), hq), device=dev) if head is None else head
    aqf = torch.empty((frames,), device=dev) if aqf is None else aqf
    dummy = torch.empty(0, device=dev)
    args, keepalive = make_args(q, k, k, cu_seqlens, n_vis, tokens_per_frame, tile, [0], [], dummy, dummy,
                                softmax_scale)
    _check(lib.evisel_coarse_evidence(ctypes.byref(args), ws.ptr, int(block), keep.data_ptr(),
                                      tok.data_ptr() if tok.numel() else None,
                                      frame.data_ptr() if frame.numel() else None, head.data_ptr(),
                                      aqf.data_ptr() if aqf.numel() else None, int(bool(accumulate)),
                                      _stream_handle(stream)))
    del keepalive
    return tok, frame, head, aqf
