"""GPU parity of the top-p block retention (evisel_topp_mask) against
oracle.topp.retained_blocks (float64 block means and logits, Eq. 7-9),
through the C ABI.

Several sets are correct where block logits (nearly) tie, so each GPU set is
checked against the oracle's p with the retention rule's four properties: it
holds the row's own block and blocks of H_i only; its mass reaches tau_p; it is
minimal (without its least block the mass is below tau_p); and it is a top set
(no dropped block has a larger p). Each property is allowed the error of the
GPU's logits, bounded per block from its arithmetic (_logit_bounds): the block
mean summed in fp32 and rounded to bf16 (the tensor cores' operand type), the
q . k_bar products accumulated in fp32, and the fp32 scaling; and the error of
its fp32 mass sums. The tile union is checked bit for bit against the union of
the GPU's own sets, and, read as a mask, it drives the probe, whose rows match
the oracle.
"""
import math

import numpy as np
import pytest

import oracle
from paper_2608_05780_gb300 import _binding as B
from paper_2608_05780_gb300 import workloads as wl
from gpu_helpers import check_lse, check_o, to_device

pytestmark = pytest.mark.gpu

U32 = 2.0 ** -24     # fp32 unit roundoff
U16 = 2.0 ** -9      # bf16 unit roundoff (round to nearest even)


def _logit_bounds(q, k, cu, n_vis, block, rows):
    """{(h, row): eps over the row's H_i}: a bound on |g_gpu - g| (natural-log
    units) for every block of H_i, from the builder's arithmetic:
      k_bar32 = fp32 sum of the block's n bf16 keys / n:
                |k_bar32 - k_bar| <= n U32 mean|k|                     (a)
      k~      = bf16(k_bar32): |k~ - k_bar32| <= U16 |k_bar32|          (b)
      S       = sum_d q_d k~_d, bf16 products exact in fp32, accumulated in
                fp32 (one rounding of at most 2 U32 per addition, whatever
                the order): |S - q.k~| <= 2 d U32 sum_d |q_d k~_d|       (c)
      x       = S scale log2(e) in fp32, then u = max - x: a few roundings of
                at most U32 relative to the row's largest |g|            (d)
    so eps_j = scale (sum_d |q_d| delta_jd + 2 d U32 sum_d |q_d| (|k_bar_jd|
    + delta_jd)) + 8 U32 max_j |g_j|, with delta_jd = (a) + U16 (|k_bar_jd| + (a))."""
    q = np.asarray(q, np.float64)
    k = np.asarray(k, np.float64)
    n, hq, d = q.shape
    gq = hq // k.shape[1]
    scale = 1.0 / math.sqrt(d)
    cu = np.asarray(cu)
    out = {}
    for row in rows:
        b = int(np.searchsorted(cu, row, side="right") - 1)
        s0, s1, nv = int(cu[b]), int(cu[b + 1]), int(n_vis[b])
        layout = oracle.block_layout(nv, s1 - s0 - nv, block)
        ends = np.array([s + ln for s, ln in layout])
        hist = np.nonzero(ends <= row - s0)[0]
        if hist.size == 0:
            for h in range(hq):
                out[(h, int(row))] = np.zeros(0)
            continue
        kv = k[s0:s1]
        kbar = np.stack([kv[layout[j][0]:layout[j][0] + layout[j][1]].mean(axis=0) for j in hist])
        mabs = np.stack([np.abs(kv[layout[j][0]:layout[j][0] + layout[j][1]]).mean(axis=0) for j in hist])
        lens = np.array([layout[j][1] for j in hist], np.float64)[:, None, None]
        a = lens * U32 * mabs
        delta = a + U16 * (np.abs(kbar) + a)
        for h in range(hq):
            qa = np.abs(q[row, h])
            g = scale * (kbar[:, h // gq] @ q[row, h])
            eps = scale * (delta[:, h // gq] @ qa + 2 * d * U32 * ((np.abs(kbar[:, h // gq]) + delta[:, h // gq]) @ qa))
            out[(h, int(row))] = eps + 8 * U32 * np.abs(g).max()
    return out


def _gpu_sets(ev, probe, block, tau, rows):
    import torch
    cfg = probe.cfg
    q, k, v = to_device(probe)
    keep, uni, ws = ev.evisel_topp_mask(q, k, probe.cu_seqlens, probe.n_vis, cfg.tokens_per_frame, cfg.tile,
                                        block, tau)
    torch.cuda.synchronize()
    assert ev.evisel_status(ws) == 0
    bits = keep[:, :, torch.as_tensor(rows, device="cuda")].cpu().numpy().view(np.uint32)   # [hq, W, len(rows)]
    ws.free()
    sets = {}
    for h in range(bits.shape[0]):
        for r, row in enumerate(rows):
            ids = [w * 32 + j for w in range(bits.shape[1]) for j in range(32) if (int(bits[h, w, r]) >> j) & 1]
            sets[(h, int(row))] = ids
    return sets, keep, uni


def _check_sets(gpu, probs, bounds, cu, n_vis, block, tau, label):
    """The retention rule's properties, each allowed the logit bound eps of
    the blocks involved: a logit off by at most e moves p by a factor within
    exp(+-2 e_max), and the builder's fp32 sums of 2^x over |H_i| blocks (x
    with ex2.approx, relative error below 2^-21) add at most eta of mass."""
    cu = np.asarray(cu)
    worst = -math.inf
    for (h, row), ids in gpu.items():
        hist, p = probs[(h, row)]
        eps = bounds[(h, row)]
        b = int(np.searchsorted(cu, row, side="right") - 1)
        pos = row - int(cu[b])
        nv = int(n_vis[b])
        own = pos // block if pos < nv else nv // block + (pos - nv) // block
        assert own in ids, (label, h, row, "own block")
        s = [j for j in ids if j != own]
        assert set(s) <= set(int(x) for x in hist), (label, h, row, "outside H_i")
        if hist.size == 0:
            assert not s
            continue
        kept = np.isin(hist, s)
        mass = p[kept].sum()
        e_max = float(eps.max())
        eta = 2.0 ** -21 + (hist.size + 2) * 2 * U32
        lo = tau * math.exp(-2 * e_max) - eta
        hi = tau * math.exp(2 * e_max) + eta + 2 * e_max
        assert mass >= lo, (label, h, row, "mass", mass, lo)
        assert mass - p[kept].min() < hi, (label, h, row, "not minimal", mass, p[kept].min(), hi)
        if (~kept).any():
            # top set: every kept block's logit, raised by its bound, reaches every
            # dropped block's logit lowered by its own (log p differs from g by a constant)
            with np.errstate(divide="ignore"):
                lp = np.log(p)
            worst = max(worst, float(np.max(lp[~kept] - eps[~kept]) - np.min(lp[kept] + eps[kept])))
            assert np.min(lp[kept] + eps[kept]) >= np.max(lp[~kept] - eps[~kept]), (label, h, row, "not a top set")
    return worst


def _all_rows(probe):
    return np.arange(int(probe.cu_seqlens[-1]))


@pytest.mark.parametrize("name,block,tau", [("tiny", 16, 0.97), ("single", 16, 0.97), ("single", 16, 0.5)])
def test_topp_sets_small(cuda_lib, name, block, tau):
    probe = wl.make_probe(wl.CONFIGS[name])
    rows = _all_rows(probe)
    gpu, _, _ = _gpu_sets(cuda_lib, probe, block, tau, rows)
    _, probs = oracle.retained_blocks(probe.q, probe.k, probe.cu_seqlens, probe.n_vis, block, tau, rows=rows)
    bounds = _logit_bounds(probe.q, probe.k, probe.cu_seqlens, probe.n_vis, block, rows)
    _check_sets(gpu, probs, bounds, probe.cu_seqlens, probe.n_vis, block, tau, name)


@pytest.mark.parametrize("name,block,n_rows", [("long65k", 64, 24), ("varlen8", 16, 24)])
def test_topp_sets_sampled(cuda_lib, name, block, n_rows):
    probe = wl.make_probe(wl.CONFIGS[name])
    rng = np.random.default_rng(3)
    n = int(probe.cu_seqlens[-1])
    rows = np.unique(np.concatenate([[0, n - 1], probe.cu_seqlens[1:-1], rng.integers(0, n, n_rows)]))
    gpu, _, _ = _gpu_sets(cuda_lib, probe, block, 0.97, rows)
    _, probs = oracle.retained_blocks(probe.q, probe.k, probe.cu_seqlens, probe.n_vis, block, 0.97, rows=rows)
    bounds = _logit_bounds(probe.q, probe.k, probe.cu_seqlens, probe.n_vis, block, rows)
    _check_sets(gpu, probs, bounds, probe.cu_seqlens, probe.n_vis, block, 0.97, name)


EDGE = {
    "planted_sharp_b32": dict(frames=(40,), n_text=(60,), npf=64, hq=4, hkv=2, d=128, tile=128, window=2, sharp=True),
    "t64_d64_b16": dict(frames=(20,), n_text=(40,), hq=6, hkv=2, d=64, tile=64, window=2),
    "varlen_mixed": dict(frames=(3, 0, 17, 8), n_text=(12, 40, 0, 130), hq=4, hkv=2, d=128, tile=128, window=2),
}


@pytest.mark.parametrize("name,block,tau", [("planted_sharp_b32", 32, 0.97), ("planted_sharp_b32", 64, 0.3),
                                            ("t64_d64_b16", 16, 0.9), ("varlen_mixed", 16, 0.97),
                                            ("varlen_mixed", 16, 1.0)])
def test_topp_edge_cases(cuda_lib, name, block, tau):
    from test_gpu_parity import _custom
    probe = _custom(**EDGE[name])
    rows = _all_rows(probe)
    gpu, _, _ = _gpu_sets(cuda_lib, probe, block, tau, rows)
    _, probs = oracle.retained_blocks(probe.q, probe.k, probe.cu_seqlens, probe.n_vis, block, tau, rows=rows)
    bounds = _logit_bounds(probe.q, probe.k, probe.cu_seqlens, probe.n_vis, block, rows)
    _check_sets(gpu, probs, bounds, probe.cu_seqlens, probe.n_vis, block, min(tau, 1.0 - 1e-6), name)


@pytest.mark.parametrize("tau", [0.97, 0.5, 1.0])
def test_topp_window_overflow(cuda_lib, tau):
    """Rows whose boundary window holds more blocks than a row's list: heads 0
    and 1 (one pair of KV group 0) have q = 0, so every block of H_i ties and
    rows with more than 32 blocks flag the pair for the radix path; heads 2-5
    keep their random q (the fast path, in the same CTAs). With all logits
    equal, S_i is the first ceil(tau |H_i|) blocks by id."""
    from test_gpu_parity import _custom
    probe = _custom(frames=(80,), n_text=(40,), npf=16, hq=6, hkv=2, d=64, tile=64, window=2, seed=11)
    probe.q[:, :2, :] = 0.0
    rows = _all_rows(probe)
    gpu, _, _ = _gpu_sets(cuda_lib, probe, 16, tau, rows)
    _, probs = oracle.retained_blocks(probe.q, probe.k, probe.cu_seqlens, probe.n_vis, 16, tau, rows=rows)
    bounds = _logit_bounds(probe.q, probe.k, probe.cu_seqlens, probe.n_vis, 16, rows)
    _check_sets(gpu, probs, bounds, probe.cu_seqlens, probe.n_vis, 16, min(tau, 1.0 - 1e-6), "overflow")
    n_long = 0
    for row in rows:
        hist, _ = probs[(0, int(row))]
        n_long += hist.size > 32
        for h in (0, 1):
            own = int(row) // 16 if row < 1280 else 80 + (int(row) - 1280) // 16
            want = list(range(math.ceil(tau * hist.size - 1e-9))) if hist.size else []
            assert sorted(set(gpu[(h, int(row))]) - {own}) == want, (tau, h, int(row))
    assert n_long > 500       # most rows take the radix path


UNION_CASES = {
    # (probe, block): blocks per key tile 8, 4, 2 and 1; tiles of 64 and 128; ragged tiles, packed videos
    "single_b16": ("single", None, 16),
    "t128_b32": (None, dict(frames=(30,), n_text=(25,), npf=32, hq=4, hkv=2, d=64, tile=128, window=2), 32),
    "t64_b16": (None, dict(frames=(23,), n_text=(30,), npf=16, hq=4, hkv=2, d=64, tile=64, window=2), 16),
    "t64_b64": (None, dict(frames=(21,), n_text=(17,), npf=64, hq=4, hkv=2, d=64, tile=64, window=2), 64),
    "t128_b64": (None, dict(frames=(3, 9, 14), n_text=(20, 0, 45), npf=64, hq=6, hkv=2, d=128, tile=128,
                            window=2), 64),
    "t128_b128": (None, dict(frames=(13, 6), n_text=(40, 9), npf=128, hq=4, hkv=1, d=128, tile=128, window=2), 128),
    # 1,280 visual blocks: the union's second chunk of 1,024 blocks
    "t128_b16_two_chunks": (None, dict(frames=(80,), n_text=(20,), npf=16, hq=4, hkv=2, d=64, tile=128, window=2), 16),
}


@pytest.mark.parametrize("case", sorted(UNION_CASES))
def test_topp_union_matches_the_sets(cuda_lib, case):
    """The tile union, bit for bit, against the union of the GPU's own sets of
    every visual row and head, folded into key tiles."""
    from test_gpu_parity import _custom
    name, custom, block = UNION_CASES[case]
    probe = wl.make_probe(wl.CONFIGS[name]) if name else _custom(**custom)
    cfg = probe.cfg
    rows = _all_rows(probe)
    gpu, _, uni = _gpu_sets(cuda_lib, probe, block, 0.6, rows)
    row_ptr, col_idx = B.tile_union_to_csr(uni, probe.n_vis, cfg.tile)
    bpt = cfg.tile // block
    r0 = 0
    for b in range(len(probe.n_vis)):
        s0, nv = int(probe.cu_seqlens[b]), int(probe.n_vis[b])
        n_vt = -(-nv // cfg.tile)
        want = [set() for _ in range(n_vt)]
        for (h, row), ids in gpu.items():
            if s0 <= row < s0 + nv:
                want[(row - s0) // cfg.tile] |= {j // bpt for j in ids if j < nv // block}
        for r in range(n_vt):
            assert sorted(want[r]) == list(col_idx[row_ptr[r0 + r]:row_ptr[r0 + r + 1]]), (case, b, r)
        r0 += n_vt


def test_topp_union_drives_the_probe(cuda_lib):
    """The tile union equals the union of the GPU's own sets; as a mask it runs the probe."""
    import torch
    probe = wl.make_probe(wl.CONFIGS["single"])
    cfg = probe.cfg
    rows = _all_rows(probe)
    gpu, keep, uni = _gpu_sets(cuda_lib, probe, 16, 0.5, rows)
    row_ptr, col_idx = B.tile_union_to_csr(uni, probe.n_vis, cfg.tile)
    # union of the sets of every visual row and head, mapped to key tiles
    n_vis = int(probe.n_vis[0])
    bpt = cfg.tile // 16
    n_vt = -(-n_vis // cfg.tile)
    want = [set() for _ in range(n_vt)]
    for (h, row), ids in gpu.items():
        if row < n_vis:
            want[row // cfg.tile] |= {j // bpt for j in ids if j < n_vis // 16}
    for r in range(n_vt):
        assert sorted(want[r]) == list(col_idx[row_ptr[r]:row_ptr[r + 1]]), r
    # the probe with this mask
    q, k, v = to_device(probe)
    o, lse, ws = cuda_lib.evisel_probe_attention(q, k, v, probe.cu_seqlens, probe.n_vis, cfg.tokens_per_frame,
                                                 cfg.tile, row_ptr, col_idx)
    torch.cuda.synchronize()
    ws.free()
    pick = np.array([0, 100, 1000, 2047, 4095, 4100, 4159])
    o_ref, lse_ref = oracle.probe_rows(probe.q, probe.k, probe.v, probe.cu_seqlens, probe.n_vis, cfg.tile, row_ptr,
                                       col_idx, pick)
    check_o(o.float().cpu().numpy()[pick], o_ref, "probe on the top-p union")
    check_lse(lse.cpu().numpy()[:, pick], lse_ref, "probe on the top-p union")


def _sets_from_keep(keep, rows, cu, n_vis, block):
    """{(h, row): retained block ids} without the own block, from keep bits."""
    import torch
    bits = keep[:, :, torch.as_tensor(rows, device=keep.device)].cpu().numpy().view(np.uint32)
    out = {}
    cu = np.asarray(cu)
    for h in range(bits.shape[0]):
        for r, row in enumerate(rows):
            b = int(np.searchsorted(cu, row, side="right") - 1)
            pos = int(row) - int(cu[b])
            nv = int(n_vis[b])
            own = pos // block if pos < nv else nv // block + (pos - nv) // block
            ids = [w * 32 + j for w in range(bits.shape[1]) for j in range(32) if (int(bits[h, w, r]) >> j) & 1]
            out[(h, int(row))] = [j for j in ids if j != own]
    return out


@pytest.mark.parametrize("name,block,tau", [("single", 16, 0.5), ("tiny", 16, 0.6)])
def test_probe_attends_only_the_retained_blocks(cuda_lib, name, block, tau):
    """Probe with the per-row masks (and the union as the tile mask) against the
    oracle restricted to the same sets: O, LSE and the evidence maps."""
    import torch
    from gpu_helpers import check_maps, np32
    probe = wl.make_probe(wl.CONFIGS[name])
    cfg = probe.cfg
    q, k, v = to_device(probe)
    keep, uni, ws = cuda_lib.evisel_topp_mask(q, k, probe.cu_seqlens, probe.n_vis, cfg.tokens_per_frame, cfg.tile,
                                              block, tau)
    row_ptr, col_idx = B.tile_union_to_csr(uni, probe.n_vis, cfg.tile)
    o, lse, ws = cuda_lib.evisel_probe_attention(q, k, v, probe.cu_seqlens, probe.n_vis, cfg.tokens_per_frame,
                                                 cfg.tile, row_ptr, col_idx, ws=ws, keep=keep, keep_block=block)
    maps = cuda_lib.evisel_evidence_reduce(ws, cfg.hq, probe.n_vis, cfg.tokens_per_frame, len(probe.n_vis))
    torch.cuda.synchronize()
    assert cuda_lib.evisel_status(ws) == 0
    n = int(probe.cu_seqlens[-1])
    rows = np.arange(n)
    kept = _sets_from_keep(keep, rows, probe.cu_seqlens, probe.n_vis, block)
    pick = np.unique(np.concatenate([np.arange(0, n, max(1, n // 40)), np.arange(n - 8, n)]))
    o_ref, lse_ref = oracle.probe_rows_topp(probe.q, probe.k, probe.v, probe.cu_seqlens, probe.n_vis, block, kept,
                                            pick)
    check_o(o.float().cpu().numpy()[pick], o_ref, f"{name} top-p probe")
    check_lse(lse.cpu().numpy()[:, pick], lse_ref, f"{name} top-p probe")
    want = oracle.evidence_topp(probe.q, probe.k, probe.cu_seqlens, probe.n_vis, cfg.tokens_per_frame, block, kept)
    check_maps([np32(m) for m in maps], list(want), probe, label=f"{name} top-p evidence")
    ws.free()


def test_keep_refused_where_it_does_not_apply(cuda_lib):
    import torch
    probe = wl.make_probe(wl.CONFIGS["tiny"])
    cfg = probe.cfg
    q, k, v = to_device(probe)
    keep, uni, ws = cuda_lib.evisel_topp_mask(q, k, probe.cu_seqlens, probe.n_vis, cfg.tokens_per_frame, cfg.tile,
                                              16, 0.9)
    row_ptr, col_idx = B.tile_union_to_csr(uni, probe.n_vis, cfg.tile)
    with pytest.raises(B.EviselError):
        cuda_lib.evisel_probe_attention(q, k, v, probe.cu_seqlens, probe.n_vis, cfg.tokens_per_frame, cfg.tile,
                                        row_ptr, col_idx, ws=ws, keep=keep, keep_block=16, cross_frame=True)
    o, lse, ws = cuda_lib.evisel_probe_attention(q, k, v, probe.cu_seqlens, probe.n_vis, cfg.tokens_per_frame,
                                                 cfg.tile, row_ptr, col_idx, ws=ws, keep=keep, keep_block=16)
    with pytest.raises(B.EviselError):
        cuda_lib.evisel_intra_frame_evidence(q, k, v, probe.cu_seqlens, probe.n_vis, cfg.tokens_per_frame, cfg.tile,
                                             row_ptr, col_idx, o, lse, ws)
    torch.cuda.synchronize()
    ws.free()


@pytest.mark.parametrize("name,block,tau", [("single", 16, 0.5), ("tiny", 16, 0.9)])
def test_coarse_evidence_matches_oracle(cuda_lib, name, block, tau):
    """Evidence of the coarse map (Eq. 10-11) on the GPU's own retained sets
    against the oracle taken with the same sets and float64 block means (Eq. 7),
    at the maps' tolerances."""
    import torch
    from gpu_helpers import check_maps, np32
    probe = wl.make_probe(wl.CONFIGS[name])
    cfg = probe.cfg
    q, k, v = to_device(probe)
    keep, uni, ws = cuda_lib.evisel_topp_mask(q, k, probe.cu_seqlens, probe.n_vis, cfg.tokens_per_frame, cfg.tile,
                                              block, tau)
    maps = cuda_lib.evisel_coarse_evidence(q, k, probe.cu_seqlens, probe.n_vis, cfg.tokens_per_frame, cfg.tile,
                                           block, keep, ws)
    torch.cuda.synchronize()
    assert cuda_lib.evisel_status(ws) == 0
    n = int(probe.cu_seqlens[-1])
    text_rows = np.concatenate([np.arange(int(probe.cu_seqlens[b]) + int(probe.n_vis[b]), int(probe.cu_seqlens[b + 1]))
                                for b in range(len(probe.n_vis))])
    kept = _sets_from_keep(keep, text_rows, probe.cu_seqlens, probe.n_vis, block)
    want = oracle.coarse_evidence(probe.q, probe.k, probe.cu_seqlens, probe.n_vis, cfg.tokens_per_frame, block, kept)
    check_maps([np32(m) for m in maps], list(want), probe, label=f"{name} coarse evidence")
    # accumulate: a second call adds the same maps
    maps2 = cuda_lib.evisel_coarse_evidence(q, k, probe.cu_seqlens, probe.n_vis, cfg.tokens_per_frame, cfg.tile,
                                            block, keep, ws, tok=maps[0].clone(), frame=maps[1].clone(),
                                            head=maps[2].clone(), aqf=maps[3].clone(), accumulate=True)
    check_maps([np32(m) for m in maps2], [2 * w for w in want], probe, label=f"{name} coarse x2")
    ws.free()


def test_topp_sparse_regime_long(cuda_lib):
    """The 65K probe with concentrated attention (long65k_sparse: clustered
    keys and queries), where tau_p = 0.97 keeps a small share of each row's
    history, as the retention rule intends. Sampled rows' sets against the
    float64 oracle; the probe on the tile union with the per-row bits against
    the oracle restricted to the GPU's own sets, on the same rows."""
    import torch
    probe = wl.make_probe(wl.CONFIGS["long65k_sparse"])
    cfg = probe.cfg
    block, tau = cfg.tokens_per_frame, 0.97
    n = int(probe.cu_seqlens[-1])
    rng = np.random.default_rng(5)
    rows = np.unique(np.concatenate([[0, 1, 127, 128, n - 1, n - 128, int(probe.n_vis[0])], rng.integers(0, n, 24)]))
    gpu, keep, uni = _gpu_sets(cuda_lib, probe, block, tau, rows)
    _, probs = oracle.retained_blocks(probe.q, probe.k, probe.cu_seqlens, probe.n_vis, block, tau, rows=rows)
    bounds = _logit_bounds(probe.q, probe.k, probe.cu_seqlens, probe.n_vis, block, rows)
    _check_sets(gpu, probs, bounds, probe.cu_seqlens, probe.n_vis, block, tau, "long65k_sparse")
    share = [len(ids) / probs[key][0].size for key, ids in gpu.items() if probs[key][0].size >= 64]
    assert np.median(share) < 0.1, f"not the sparse regime: median kept share {np.median(share):.3f}"
    row_ptr, col_idx = B.tile_union_to_csr(uni, probe.n_vis, cfg.tile)
    q, k, v = to_device(probe)
    o, lse, ws = cuda_lib.evisel_probe_attention(q, k, v, probe.cu_seqlens, probe.n_vis, cfg.tokens_per_frame,
                                                 cfg.tile, row_ptr, col_idx, keep=keep, keep_block=block)
    torch.cuda.synchronize()
    assert cuda_lib.evisel_status(ws) == 0
    ws.free()
    kept = _sets_from_keep(keep, rows, probe.cu_seqlens, probe.n_vis, block)
    o_ref, lse_ref = oracle.probe_rows_topp(probe.q, probe.k, probe.v, probe.cu_seqlens, probe.n_vis, block, kept,
                                            rows)
    check_o(o.float().cpu().numpy()[rows], o_ref, "long65k_sparse probe on the top-p masks")
    check_lse(lse.cpu().numpy()[:, rows], lse_ref, "long65k_sparse probe on the top-p masks")
