"""The entry point that allocates nothing (evisel_probe_evidence_noalloc).

It is meant for callers that cannot let the library call cudaMalloc -- servers
that hand all device memory to their own pool, or serving paths where an
allocation is not acceptable. It keeps its scratch in a fixed static device
array, so these tests check that its results match the workspace path
(evisel_probe_attention + evisel_evidence_reduce) within the parity tolerances
on two calls in a row (the second call reuses the array the first one left
behind), and that a problem too large for the array is refused up front.

This file is named to be collected last.
"""
import ctypes

import numpy as np
import pytest

from paper_2608_05780_gb300 import _binding as B
from paper_2608_05780_gb300 import workloads as wl
from paper_2608_05780_gb300.build import build


def test_noalloc_refuses_oversized_problem_before_any_launch():
    """The 65,664-token probe needs ~1 GB of scratch: refused with ENOMEM, no GPU needed."""
    build()
    lib = B.load()
    cfg = wl.CONFIGS["long65k"]
    row_ptr, col_idx = wl.build_mask(cfg)
    fake = 0x7F0000000000           # never dereferenced: the size check comes first
    a = B.ProbeArgs()
    keep = []

    def arr(x):
        x = np.ascontiguousarray(np.asarray(x, dtype=np.int32))
        keep.append(x)
        return x.ctypes.data_as(ctypes.POINTER(ctypes.c_int32))
    a.num_videos = 1
    a.cu_seqlens_h = arr([0, cfg.n_tot])
    a.n_vis_h = arr([cfg.n_vis[0]])
    a.tokens_per_frame = cfg.tokens_per_frame
    a.hq, a.hkv, a.head_dim, a.tile = cfg.hq, cfg.hkv, cfg.head_dim, cfg.tile
    a.softmax_scale = 0.0
    a.q = a.k = a.v = a.o = a.lse = fake
    a.mask_row_ptr_h = arr(row_ptr)
    a.mask_col_idx_h = arr(col_idx)
    status = ctypes.c_int(123)
    rc = lib.evisel_probe_evidence_noalloc(ctypes.byref(a), fake, fake, fake, fake, 0, None, ctypes.byref(status))
    assert rc == -5
    msg = lib.evisel_last_error().decode()
    assert "scratch" in msg and str(B.NOALLOC_SCRATCH_BYTES) in msg
    assert status.value == 123      # nothing ran


@pytest.mark.gpu
@pytest.mark.parametrize("name", ["tiny", "single"])
def test_noalloc_matches_workspace_path_twice(cuda_lib, name):
    import torch
    from gpu_helpers import HEAD_REL, LSE_ABS, MAP_ABS, check_o, run_cuda, to_device

    probe = wl.make_probe(wl.CONFIGS[name])
    cfg = probe.cfg
    ref, ws = run_cuda(cuda_lib, probe)
    ws.free()
    q, k, v = to_device(probe)
    n, hq, d = q.shape
    total_vis = int(np.sum(probe.n_vis))
    frames = total_vis // cfg.tokens_per_frame
    for call in range(2):
        o = torch.full((n, hq, d), float("nan"), dtype=torch.bfloat16, device="cuda")
        lse = torch.full((hq, n), float("nan"), device="cuda")
        tok = torch.full((hq, total_vis), float("nan"), device="cuda")
        frame = torch.full((hq, frames), float("nan"), device="cuda")
        head = torch.full((1, hq), float("nan"), device="cuda")
        aqf = torch.full((frames,), float("nan"), device="cuda")
        status = B.evisel_probe_evidence_noalloc(q, k, v, probe.cu_seqlens, probe.n_vis, cfg.tokens_per_frame,
                                                 cfg.tile, probe.row_ptr, probe.col_idx, o, lse, tok, frame, head,
                                                 aqf)
        assert status == 0, f"call {call}: device status {status}"
        check_o(o.float().cpu().numpy(), ref["o"].double().cpu().numpy(), f"{name} call {call}")
        assert np.abs(lse.cpu().numpy() - ref["lse"].cpu().numpy()).max() <= LSE_ABS
        # raw maps: token, frame and A_qf entries within MAP_ABS, the head map within HEAD_REL (relative)
        for got, want, rel in ((tok, ref["tok"], False), (frame, ref["frame"], False), (head, ref["head"], True),
                               (aqf, ref["aqf"], False)):
            g, w = got.cpu().numpy().astype(np.float64), want.cpu().numpy().astype(np.float64)
            err = np.abs(g - w) / np.maximum(np.abs(w), 1e-30) if rel else np.abs(g - w)
            bound = HEAD_REL if rel else MAP_ABS
            assert np.all(np.isfinite(err)) and err.max() <= bound, f"{name} call {call}: map error {err.max()}"
