"""GPU parity of the intra-frame cue A_if (evisel_intra_frame_evidence) against
oracle.intra_frame, through the C ABI, on the seeded workloads and the edge
cases of the probe (ragged tiles, 64-token tiles, d = 64, N_v = 4 / 16 / 64,
packed videos with and without visual tokens, sharp logits).

Tolerance: A_if = mean_h exp(s - LSE) with the probe's own fp32 LSE, so its
relative error is that of exp(-LSE) -- at most the LSE bound (1e-3) -- plus
fp32 logit and ex2 rounding: |gpu - oracle| <= 2e-3 * oracle + 1e-6 per entry.
The 65,664-token probe and the packed 8-video batch are compared on sampled
frames (the oracle evaluates those frames' rows only).
"""
import numpy as np
import pytest

import oracle
from paper_2608_05780_gb300 import workloads as wl
from gpu_helpers import to_device

pytestmark = pytest.mark.gpu

RTOL = 2e-3
ATOL = 1e-6


def _gpu_aif(ev, probe, out=None, accumulate=False):
    import torch
    cfg = probe.cfg
    q, k, v = to_device(probe)
    o, lse, ws = ev.evisel_probe_attention(q, k, v, probe.cu_seqlens, probe.n_vis, cfg.tokens_per_frame, cfg.tile,
                                           probe.row_ptr, probe.col_idx)
    aif = ev.evisel_intra_frame_evidence(q, k, v, probe.cu_seqlens, probe.n_vis, cfg.tokens_per_frame, cfg.tile,
                                         probe.row_ptr, probe.col_idx, o, lse, ws, aif=out, accumulate=accumulate)
    torch.cuda.synchronize()
    assert ev.evisel_status(ws) == 0
    ws.free()
    return aif.cpu().numpy().astype(np.float64)


def _check(got, want, label):
    assert got.shape == want.shape, (got.shape, want.shape)
    assert np.all(np.isfinite(got)), f"{label}: non-finite A_if"
    err = np.abs(got - want)
    bound = RTOL * np.abs(want) + ATOL
    worst = np.unravel_index(np.argmax(err - bound), err.shape)
    assert np.all(err <= bound), f"{label}: A_if error {err[worst]:.3e} at {worst} (want {want[worst]:.6f})"


def _oracle_aif(probe, frames=None):
    cfg = probe.cfg
    return oracle.intra_frame(probe.q, probe.k, probe.cu_seqlens, probe.n_vis, cfg.tokens_per_frame, cfg.tile,
                              probe.row_ptr, probe.col_idx, frames=frames)


@pytest.mark.parametrize("name", ["tiny", "single"])
def test_intra_frame_full(cuda_lib, name):
    probe = wl.make_probe(wl.CONFIGS[name])
    _check(_gpu_aif(cuda_lib, probe), _oracle_aif(probe), name)


@pytest.mark.parametrize("name,n_frames", [("long65k", 12), ("varlen8", 12)])
def test_intra_frame_sampled(cuda_lib, name, n_frames):
    probe = wl.make_probe(wl.CONFIGS[name])
    total = int(np.sum(probe.n_vis)) // probe.cfg.tokens_per_frame
    rng = np.random.default_rng(5)
    frames = np.unique(np.concatenate([[0, total - 1], rng.choice(total, n_frames, replace=False)]))
    got = _gpu_aif(cuda_lib, probe)
    _check(got[frames], _oracle_aif(probe, frames), name)


EDGE = {
    "ragged_t128_d128": dict(frames=(44,), n_text=(77,), hq=8, hkv=2, d=128, tile=128, window=3),
    "t64_d128": dict(frames=(23,), n_text=(70,), hq=4, hkv=2, d=128, tile=64, window=3),
    "odd_group_t64_d64": dict(frames=(20,), n_text=(40,), hq=6, hkv=2, d=64, tile=64, window=2),
    "npf64": dict(frames=(9,), n_text=(40,), npf=64, hq=4, hkv=2, d=128, tile=128, window=2),
    "npf4": dict(frames=(70,), n_text=(20,), npf=4, hq=4, hkv=2, d=64, tile=64, window=2),
    "varlen_mixed": dict(frames=(3, 0, 17, 8), n_text=(12, 40, 0, 130), hq=4, hkv=2, d=128, tile=128, window=2),
    "sharp": dict(frames=(40,), n_text=(60,), hq=4, hkv=2, d=128, tile=128, window=4, sharp=True),
}


@pytest.mark.parametrize("name", sorted(EDGE))
def test_intra_frame_edge_cases(cuda_lib, name):
    from test_gpu_parity import _custom
    probe = _custom(**EDGE[name])
    _check(_gpu_aif(cuda_lib, probe), _oracle_aif(probe), name)


def _probe(name):
    if name in EDGE:
        from test_gpu_parity import _custom
        return _custom(**EDGE[name])
    return wl.make_probe(wl.CONFIGS[name])


@pytest.mark.parametrize("name", ["tiny", "npf64"])
def test_intra_frame_accumulates(cuda_lib, name):
    import torch
    probe = _probe(name)
    want = _oracle_aif(probe)
    base = torch.full(want.shape, 0.25, dtype=torch.float32, device="cuda")
    _check(_gpu_aif(cuda_lib, probe, out=base, accumulate=True), want + 0.25, f"accumulate {name}")


@pytest.mark.parametrize("name", ["single", "npf64", "npf4"])
def test_intra_frame_overwrites(cuda_lib, name):
    """Without accumulate every entry is written, the zeros above the diagonal included."""
    import torch
    probe = _probe(name)
    want = _oracle_aif(probe)
    out = torch.full(want.shape, float("nan"), dtype=torch.float32, device="cuda")
    _check(_gpu_aif(cuda_lib, probe, out=out), want, f"overwrite {name}")


def test_intra_frame_many_videos(cuda_lib):
    """40 packed videos of 0-9 frames (fewer 128-row blocks than SMs, empty videos between)."""
    from test_gpu_parity import _custom
    rng = np.random.default_rng(11)
    frames = tuple(int(f) for f in rng.integers(0, 10, size=40))
    n_text = tuple(int(t) for t in rng.integers(1, 40, size=40))
    probe = _custom(frames=frames, n_text=n_text, hq=4, hkv=2, d=128, tile=128, window=2)
    _check(_gpu_aif(cuda_lib, probe), _oracle_aif(probe), "many videos")
