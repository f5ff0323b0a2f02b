"""GPU parity of the cross-frame cue A_ff and E_ff (evisel_cross_frame_evidence)
against oracle.cross_frame / frame_mass_rows / e_ff, through the C ABI, on the
seeded workloads and the probe's edge cases (ragged tiles, 64-token tiles,
d = 64, N_v = 16 / 64, packed videos with and without visual tokens, sharp
logits).

Tolerance: an A_ff entry is a sum of exp2(partial - LSE log2 e) over heads and
rows, each partial the fp32 log2 of the frame's fp32 probability sum and LSE
the probe's own fp32 normaliser; the relative error is that of exp(-LSE) (at
most the LSE bound, 1e-3) plus fp32 rounding, so |gpu - oracle| <=
2e-3 |oracle| + 1e-6 per entry, and the same for E_ff (sums of A_ff entries).
The 65,664-token probe and the packed 8-video batch are compared on sampled
query frames; their E_ff is checked against e_ff applied to the GPU's own A_ff.
"""
import numpy as np
import pytest

import oracle
from paper_2608_05780_gb300 import workloads as wl
from gpu_helpers import to_device

pytestmark = pytest.mark.gpu

RTOL = 2e-3
ATOL = 1e-6


def _gpu(ev, probe, aff=None, eff=None, accumulate=False, with_probe=False):
    import torch
    cfg = probe.cfg
    q, k, v = to_device(probe)
    o, lse, ws = ev.evisel_probe_attention(q, k, v, probe.cu_seqlens, probe.n_vis, cfg.tokens_per_frame, cfg.tile,
                                           probe.row_ptr, probe.col_idx, cross_frame=True)
    aff, eff = ev.evisel_cross_frame_evidence(q, k, v, probe.cu_seqlens, probe.n_vis, cfg.tokens_per_frame,
                                              cfg.tile, probe.row_ptr, probe.col_idx, o, lse, ws, aff=aff, eff=eff,
                                              accumulate=accumulate)
    torch.cuda.synchronize()
    assert ev.evisel_status(ws) == 0
    ws.free()
    out = (aff.cpu().numpy().astype(np.float64), eff.cpu().numpy().astype(np.float64))
    if with_probe:
        out += (o.float().cpu().numpy(), lse.cpu().numpy())
    return out


def _blocks(flat, probe):
    """Splits the packed A_ff into the videos' [(T-1), (T-1)] blocks."""
    t = np.asarray(probe.n_vis) // probe.cfg.tokens_per_frame
    out, off = [], 0
    for tb in t:
        n = max(int(tb) - 1, 0)
        out.append(flat[off:off + n * n].reshape(n, n))
        off += n * n
    assert off == flat.size
    return out


def _check(got, want, label):
    assert got.shape == want.shape, (label, got.shape, want.shape)
    assert np.all(np.isfinite(got)), f"{label}: non-finite"
    err = np.abs(got - want)
    bound = RTOL * np.abs(want) + ATOL
    if err.size:
        worst = np.unravel_index(np.argmax(err - bound), err.shape)
        assert np.all(err <= bound), f"{label}: error {err[worst]:.3e} at {worst} (want {want[worst]:.6e})"


def _oracle(probe):
    cfg = probe.cfg
    return oracle.cross_frame(probe.q, probe.k, probe.cu_seqlens, probe.n_vis, cfg.tokens_per_frame, cfg.tile,
                              probe.row_ptr, probe.col_idx)


def _custom(**kw):
    from test_gpu_parity import _custom as c
    return c(**kw)


@pytest.mark.parametrize("name", ["tiny", "single"])
def test_cross_frame_full(cuda_lib, name):
    probe = wl.make_probe(wl.CONFIGS[name])
    aff, eff = _gpu(cuda_lib, probe)
    waff, weff = _oracle(probe)
    for b, (g, w) in enumerate(zip(_blocks(aff, probe), waff)):
        _check(g, w, f"{name} A_ff video {b}")
    _check(eff, weff, f"{name} E_ff")


@pytest.mark.parametrize("name,n_frames", [("long65k", 6), ("varlen8", 8)])
def test_cross_frame_sampled(cuda_lib, name, n_frames):
    probe = wl.make_probe(wl.CONFIGS[name])
    cfg = probe.cfg
    npf = cfg.tokens_per_frame
    t = np.asarray(probe.n_vis) // npf
    fr_off = np.concatenate([[0], np.cumsum(t)])
    aff, eff = _gpu(cuda_lib, probe)
    blocks = _blocks(aff, probe)
    rng = np.random.default_rng(9)
    # query frames other than a video's first one (those have no A_ff row)
    cand = np.concatenate([np.arange(fr_off[b] + 1, fr_off[b + 1]) for b in range(len(t))])
    frames = np.unique(np.concatenate([[cand[0], cand[-1]], rng.choice(cand, n_frames, replace=False)]))
    rows = oracle.frame_mass_rows(probe.q, probe.k, probe.cu_seqlens, probe.n_vis, npf, cfg.tile, probe.row_ptr,
                                  probe.col_idx, frames)
    for f, want in zip(frames, rows):
        b = int(np.searchsorted(fr_off, f, side="right") - 1)
        a = int(f - fr_off[b])
        _check(blocks[b][a - 1, :a], want[:a], f"{name} A_ff frame {f}")
        assert np.all(blocks[b][a - 1, a:] == 0.0)
    # E_ff is the deterministic function e_ff of A_ff
    _check(eff, oracle.e_ff(blocks, t), f"{name} E_ff")


EDGE = {
    "ragged_t128_d128": dict(frames=(44,), n_text=(77,), hq=8, hkv=2, d=128, tile=128, window=3),
    "t64_d128": dict(frames=(23,), n_text=(70,), hq=4, hkv=2, d=128, tile=64, window=3),
    "odd_group_t64_d64": dict(frames=(20,), n_text=(40,), hq=6, hkv=2, d=64, tile=64, window=2),
    "npf64": dict(frames=(9,), n_text=(40,), npf=64, hq=4, hkv=2, d=128, tile=128, window=2),
    "npf32_extra": dict(frames=(40,), n_text=(16,), npf=32, hq=4, hkv=2, d=128, tile=128, window=2, extra=2),
    "npf128_two_spans": dict(frames=(6,), n_text=(20,), npf=128, hq=4, hkv=2, d=128, tile=128, window=3),
    "npf64_t64_d64": dict(frames=(12,), n_text=(24,), npf=64, hq=4, hkv=2, d=64, tile=64, window=3),
    "varlen_mixed": dict(frames=(3, 0, 17, 8, 1), n_text=(12, 40, 0, 130, 9), hq=4, hkv=2, d=128, tile=128,
                         window=2),
    "sharp": dict(frames=(40,), n_text=(60,), hq=4, hkv=2, d=128, tile=128, window=4, sharp=True),
}


@pytest.mark.parametrize("name", sorted(EDGE))
def test_cross_frame_edge_cases(cuda_lib, name):
    probe = _custom(**EDGE[name])
    aff, eff = _gpu(cuda_lib, probe)
    waff, weff = _oracle(probe)
    for b, (g, w) in enumerate(zip(_blocks(aff, probe), waff)):
        _check(g, w, f"{name} A_ff video {b}")
    _check(eff, weff, f"{name} E_ff")


def test_cross_frame_overwrites_and_accumulates(cuda_lib):
    import torch
    probe = _custom(**EDGE["npf64"])
    waff, weff = _oracle(probe)
    t = np.asarray(probe.n_vis) // probe.cfg.tokens_per_frame
    n = int(np.sum(np.maximum(t - 1, 0) ** 2))
    aff = torch.full((n,), float("nan"), device="cuda")
    eff = torch.full((int(t.sum()),), float("nan"), device="cuda")
    got_aff, got_eff = _gpu(cuda_lib, probe, aff=aff, eff=eff)
    _check(_blocks(got_aff, probe)[0], waff[0], "overwrite A_ff")
    _check(got_eff, weff, "overwrite E_ff")
    base = torch.full((n,), 0.5, device="cuda")
    got_aff, got_eff = _gpu(cuda_lib, probe, aff=base, accumulate=True)
    _check(_blocks(got_aff, probe)[0], waff[0] + 0.5, "accumulate A_ff")
    # E_ff is recomputed from the accumulated A_ff (its entries b < a: the lower triangle with the diagonal)
    _check(got_eff, oracle.e_ff([waff[0] + 0.5 * np.tril(np.ones_like(waff[0]))], t), "accumulate E_ff")


def test_probe_with_cross_frame_partials_still_matches(cuda_lib):
    """The probe instantiation that keeps the partials leaves O and LSE as the oracle has them."""
    probe = wl.make_probe(wl.CONFIGS["single"])
    cfg = probe.cfg
    _, _, o, lse = _gpu(cuda_lib, probe, with_probe=True)
    want_o, want_lse = oracle.probe(probe.q, probe.k, probe.v, probe.cu_seqlens, probe.n_vis, cfg.tile,
                                    probe.row_ptr, probe.col_idx)
    assert np.max(np.abs(lse - want_lse)) <= 1e-3
    diff = o.astype(np.float64) - want_o
    assert np.max(np.abs(diff)) <= 2e-2
    assert np.linalg.norm(diff) / np.linalg.norm(want_o) <= 5e-3
