"""GPU parity: the sm_103a path (through the C ABI) against the float64 oracle.

Small workloads are compared on every output; the full-size workloads (65,664
tokens; 8 packed videos; 28 layers) are compared on sampled rows of O/LSE (the
oracle computes them one by one) and on the complete evidence maps (which only
need the text rows). Edge cases: ragged visual and text tiles, text shorter than
a tile, a one-frame video, videos without text or without visual tokens, an
empty batch, odd query-head groups with 64-token tiles, MHA, random masks and
sharp logits that exercise the lazy rescale.
"""
import math

import numpy as np
import pytest

import oracle
from paper_2608_05780_gb300 import workloads as wl
from gpu_helpers import check_lse, check_maps, check_o, np32, oracle_maps, run_cuda, to_device

pytestmark = pytest.mark.gpu


def _full_compare(ev, probe, label):
    out, ws = run_cuda(ev, probe)
    o_ref, lse_ref = oracle.probe(probe.q, probe.k, probe.v, probe.cu_seqlens, probe.n_vis, probe.cfg.tile,
                                  probe.row_ptr, probe.col_idx)
    check_o(np32(out["o"]), o_ref, label)
    check_lse(np32(out["lse"]), lse_ref, label)
    check_maps([np32(out[k]) for k in ("tok", "frame", "head", "aqf")], oracle_maps(probe), probe, label=label)
    ws.free()


def _sampled_compare(ev, probe, rows, label, out=None):
    if out is None:
        out, ws = run_cuda(ev, probe)
        ws.free()
    o_ref, lse_ref = oracle.probe_rows(probe.q, probe.k, probe.v, probe.cu_seqlens, probe.n_vis, probe.cfg.tile,
                                       probe.row_ptr, probe.col_idx, rows)
    check_o(np32(out["o"][rows]), o_ref, label)
    check_lse(np32(out["lse"][:, rows]), lse_ref, label)
    return out


def _sample_rows(probe, per_video=24, seed=0):
    """Rows spread over each video: its first/last visual rows, a ragged tile, text rows."""
    rng = np.random.default_rng(seed)
    rows = []
    for b in range(len(probe.n_vis)):
        s0, s1 = int(probe.cu_seqlens[b]), int(probe.cu_seqlens[b + 1])
        nv = int(probe.n_vis[b])
        pick = {s0, s0 + nv - 1, s1 - 1, s0 + nv} if nv > 0 else {s0, s1 - 1}
        pick |= set(int(x) for x in rng.integers(s0, s1, per_video))
        pick |= set(int(x) for x in rng.integers(s0 + nv, s1, max(per_video // 3, 1)))
        rows += sorted(p for p in pick if s0 <= p < s1)
    return np.array(sorted(set(rows)), dtype=np.int64)


def test_tiny_full(cuda_lib):
    _full_compare(cuda_lib, wl.make_probe(wl.CONFIGS["tiny"]), "tiny")


def test_single_full(cuda_lib):
    _full_compare(cuda_lib, wl.make_probe(wl.CONFIGS["single"]), "single")


def _whole_tiles(probe):
    """{label: global rows} of whole query tiles that, over all heads, run every
    item class of the attention kernel: the visual row tile with the most kept
    kv tiles (the longest items), the first visual tile, the last visual tile
    of each video (ragged where n_vis is not a multiple of the tile), and every
    text row of each video (its kv range is split over several items whose
    partials the combine merges). All heads of a tile cover both the two-slot
    items and the one-slot item of a KV group's odd last head."""
    T = probe.cfg.tile
    counts = np.diff(probe.row_ptr)
    tiles = {}
    r0 = 0
    best = (-1, None)
    for b in range(len(probe.n_vis)):
        s0, s1, nv = int(probe.cu_seqlens[b]), int(probe.cu_seqlens[b + 1]), int(probe.n_vis[b])
        n_vt = -(-nv // T)
        for t in range(n_vt):
            if counts[r0 + t] > best[0]:
                best = (int(counts[r0 + t]), (b, t))
        if n_vt and b == 0:
            tiles[f"video {b} first visual tile"] = np.arange(s0, s0 + min(T, nv))
        if n_vt:
            tiles[f"video {b} last visual tile ({nv - (n_vt - 1) * T} rows)"] = np.arange(s0 + (n_vt - 1) * T, s0 + nv)
        if s1 > s0 + nv:
            tiles[f"video {b} text rows ({s1 - s0 - nv})"] = np.arange(s0 + nv, s1)
        r0 += n_vt
    if best[1] is not None:
        b, t = best[1]
        s0, nv = int(probe.cu_seqlens[b]), int(probe.n_vis[b])
        tiles[f"video {b} visual tile {t} ({best[0]} kv tiles)"] = np.arange(s0 + t * T, s0 + min((t + 1) * T, nv))
    return tiles


def _tile_compare(probe, out, label):
    for name, rows in _whole_tiles(probe).items():
        _sampled_compare(None, probe, rows, f"{label}: {name}", out=out)


def test_long65k_sampled_and_maps(cuda_lib):
    probe = wl.make_probe(wl.CONFIGS["long65k"])
    out, ws = run_cuda(cuda_lib, probe)
    ws.free()
    rows = _sample_rows(probe, per_video=96)
    _sampled_compare(cuda_lib, probe, rows, "long65k", out=out)
    _tile_compare(probe, out, "long65k")
    check_maps([np32(out[k]) for k in ("tok", "frame", "head", "aqf")], oracle_maps(probe), probe,
               label="long65k")


def test_varlen8_sampled_and_maps(cuda_lib):
    probe = wl.make_probe(wl.CONFIGS["varlen8"])
    out, ws = run_cuda(cuda_lib, probe)
    ws.free()
    rows = _sample_rows(probe, per_video=16)
    _sampled_compare(cuda_lib, probe, rows, "varlen8", out=out)
    _tile_compare(probe, out, "varlen8")
    check_maps([np32(out[k]) for k in ("tok", "frame", "head", "aqf")], oracle_maps(probe), probe,
               label="varlen8")


def test_depth28_accumulated_evidence(cuda_lib):
    import torch
    cfg = wl.CONFIGS["depth28"]
    mask = wl.build_mask(cfg)
    ws = None
    maps = None
    ref = None
    for layer in range(cfg.layers):
        probe = wl.make_probe(cfg, layer, mask=mask)
        out, ws = run_cuda(cuda_lib, probe, ws=ws, maps=maps, accumulate=layer > 0)
        maps = [out[k] for k in ("tok", "frame", "head", "aqf")]
        r = oracle_maps(probe)
        ref = r if ref is None else [a + b for a, b in zip(ref, r)]
        if layer in (0, cfg.layers - 1):
            rows = _sample_rows(probe, per_video=24, seed=layer)
            _sampled_compare(cuda_lib, probe, rows, f"depth28 layer {layer}", out=out)
    torch.cuda.synchronize()
    check_maps([np32(m) for m in maps], ref, probe, label="depth28 (sum of layers)")
    ws.free()


def _custom(frames, n_text, npf=16, hq=4, hkv=2, d=64, tile=64, window=2, extra=0, plant=None, seed=7,
            sharp=False, mask=None):
    cfg = wl.ProbeConfig("custom", tuple(frames), npf, tuple(n_text), hq, hkv, d, tile, window, extra=extra,
                         plant=tuple(plant) if plant else (), seed=seed, mask_seed=seed,
                         scale_inputs=not sharp)
    p = wl.make_probe(cfg, mask=mask)
    if sharp:
        # x4 keeps bf16 values exact; logits then have a std of about 16
        p.q *= 4.0
        p.k *= 4.0
    return p


EDGE_CASES = {
    # 44 frames x 16 = 704 tokens = 5 full 128-tiles + a ragged 64-token tile
    "ragged_tiles_t128_d128": dict(frames=(44,), n_text=(77,), hq=8, hkv=2, d=128, tile=128, window=3),
    "t128_d64": dict(frames=(36,), n_text=(50,), hq=4, hkv=1, d=64, tile=128, window=2),
    "t64_d128": dict(frames=(23,), n_text=(70,), hq=4, hkv=2, d=128, tile=64, window=3),
    "odd_group_t64": dict(frames=(20,), n_text=(40,), hq=6, hkv=2, d=64, tile=64, window=2),
    "mha_t128": dict(frames=(24,), n_text=(33,), hq=3, hkv=3, d=128, tile=128, window=2),
    "short_text": dict(frames=(16,), n_text=(5,), hq=4, hkv=2, d=64, tile=64, window=2),
    "one_frame": dict(frames=(1,), n_text=(9,), hq=4, hkv=2, d=64, tile=64, window=2),
    "npf64_t128": dict(frames=(9,), n_text=(40,), npf=64, hq=4, hkv=2, d=128, tile=128, window=2),
    "npf4": dict(frames=(70,), n_text=(20,), npf=4, hq=4, hkv=2, d=64, tile=64, window=2),
    "varlen_mixed": dict(frames=(3, 0, 17, 8), n_text=(12, 40, 0, 130), hq=4, hkv=2, d=128, tile=128,
                         window=2),
    "random_extra": dict(frames=(64,), n_text=(64,), hq=4, hkv=2, d=64, tile=64, window=2, extra=3),
    "sharp_rescale": dict(frames=(40,), n_text=(60,), hq=4, hkv=2, d=128, tile=128, window=4, sharp=True),
    "sharp_rescale_t64": dict(frames=(40,), n_text=(60,), hq=4, hkv=2, d=64, tile=64, window=4, sharp=True,
                              extra=2),
}


@pytest.mark.parametrize("name", sorted(EDGE_CASES))
def test_edge_case_full(cuda_lib, name):
    _full_compare(cuda_lib, _custom(**EDGE_CASES[name]), name)


def test_empty_batch(cuda_lib):
    import torch
    z = torch.zeros((0, 4, 64), dtype=torch.bfloat16, device="cuda")
    zk = torch.zeros((0, 2, 64), dtype=torch.bfloat16, device="cuda")
    o, lse, ws = cuda_lib.evisel_probe_attention(z, zk, zk, [0], [], 16, 64, [0], [])
    assert o.shape == (0, 4, 64) and lse.shape == (4, 0)
    cuda_lib.evisel_evidence_reduce(ws, 4, np.zeros(0, np.int32), 16, 0)
    assert cuda_lib.evisel_status(ws) == 0
    ws.free()


def test_workspace_reuse_and_replan(cuda_lib):
    """One workspace across different shapes; repeated calls give identical results."""
    a = _custom(frames=(30,), n_text=(20,))
    b = _custom(frames=(12, 9), n_text=(40, 3), seed=9)
    out_a1, ws = run_cuda(cuda_lib, a)
    out_b, ws = run_cuda(cuda_lib, b, ws=ws)
    out_a2, ws = run_cuda(cuda_lib, a, ws=ws)
    for k in ("o", "lse", "tok", "frame", "head", "aqf"):
        assert np.array_equal(np32(out_a1[k]), np32(out_a2[k])), k
    o_ref, lse_ref = oracle.probe(b.q, b.k, b.v, b.cu_seqlens, b.n_vis, b.cfg.tile, b.row_ptr, b.col_idx)
    check_o(np32(out_b["o"]), o_ref, "replan")
    ws.free()


def test_dense_mask_matches_sdpa(cuda_lib):
    """All causal tiles kept: the kernel equals dense causal attention (torch SDPA)."""
    import torch
    cfg = wl.ProbeConfig("dense", (40,), 16, (64,), 8, 2, 128, 128, 1000, seed=5)
    p = wl.make_probe(cfg)
    out, ws = run_cuda(cuda_lib, p)
    ws.free()
    q, k, v = to_device(p)
    ref = torch.nn.functional.scaled_dot_product_attention(
        q.float().transpose(0, 1), k.float().transpose(0, 1).repeat_interleave(4, 0),
        v.float().transpose(0, 1).repeat_interleave(4, 0), is_causal=True).transpose(0, 1)
    check_o(np32(out["o"]), ref.double().cpu().numpy(), "dense vs sdpa")
