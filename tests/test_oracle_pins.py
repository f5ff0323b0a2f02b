"""Pins of the float64 oracle against facts other than itself (CPU only).

Each test names the pin it realises:
  golden  hand-derived example (tests/golden/hand_mask_example.json)
  O1  closed form for constant keys
  O2  row mass 1 and mass conservation of the evidence maps (also sharp logits)
  O3  all-causal-tiles mask equals dense causal attention (torch SDPA, float64)
  O4  brute force, pure-Python loops, tiny varlen inputs with random masks
  O5  key-shift invariance of P, LSE shift by scale q.c
  O6  GQA equals MHA with replicated KV heads
  O7  packed varlen equals per-video runs
  O8  reductions: frame, head, A_qf from tok
  O9  planted frames rank top on the head-summed frame map
  O10 linearity of O in V
  F1-F4 the intra-frame cue A_if (closed form, dense weights, brute force, structure)
  H1-H7 top-p block retention (closed form, brute force, planted block, limits, keep-all,
        bf16 rounding of the block means, evidence with every block kept)
  C1-C3 the coarse map of Eq. 10-11 (one-token blocks and constant keys give the exact map, mass)
  G1-G5 the cross-frame cue A_ff and E_ff (closed form, mass balance with A_if, brute force,
        dense weights, a hand-worked E_ff)
"""
import json
import math
import os

import numpy as np
import pytest

import oracle
from paper_2608_05780_gb300 import workloads as wl

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def _random_case(seed, videos=((6, 5), (10, 7)), hq=4, hkv=2, d=8, tile=4, npf=2, density=0.5,
                 sharp=False):
    """Tiny varlen case: videos = ((n_vis, n_text), ...); random valid CSR."""
    rng = np.random.default_rng(seed)
    n_vis = np.array([a for a, _ in videos], np.int32)
    lens = np.array([a + b for a, b in videos])
    cu = np.concatenate([[0], np.cumsum(lens)]).astype(np.int32)
    n = int(cu[-1])
    sc = 1.0 if sharp else 1.0 / math.sqrt(d)
    q = wl.bf16_round(rng.standard_normal((n, hq, d)).astype(np.float32) * sc)
    k = wl.bf16_round(rng.standard_normal((n, hkv, d)).astype(np.float32) * sc)
    v = wl.bf16_round(rng.standard_normal((n, hkv, d)).astype(np.float32))
    row_ptr, cols = [0], []
    for nv in n_vis:
        for r in range(-(-int(nv) // tile)):
            kept = {r} | {c for c in range(r) if rng.random() < density}
            cols += sorted(kept)
            row_ptr.append(len(cols))
    return dict(q=q, k=k, v=v, cu=cu, n_vis=n_vis, tile=tile, npf=npf,
                row_ptr=np.array(row_ptr, np.int32), col_idx=np.array(cols, np.int32))


def _run(c, scale=None):
    o, lse = oracle.probe(c["q"], c["k"], c["v"], c["cu"], c["n_vis"], c["tile"], c["row_ptr"], c["col_idx"],
                          scale=scale)
    maps = oracle.evidence(c["q"], c["k"], c["cu"], c["n_vis"], c["npf"], scale=scale)
    return o, lse, maps


# ---------------------------------------------------------------- golden
def test_golden_hand_example():
    g = json.load(open(os.path.join(GOLDEN, "hand_mask_example.json")))
    n = len(g["q"])
    q = np.array(g["q"], np.float64).reshape(n, 1, 1)
    k = np.log(np.array(g["k_exp"], np.float64)).reshape(n, 1, 1)
    v = np.array(g["v"], np.float64).reshape(n, 1, 1)
    cu = np.array([0, n]); n_vis = np.array([4])
    o, lse = oracle.probe(q, k, v, cu, n_vis, g["tile"], np.array(g["row_ptr"]), np.array(g["col_idx"]),
                          scale=1.0)
    np.testing.assert_allclose(o[:, 0, 0], g["expected_o"], rtol=1e-14, atol=1e-14)
    np.testing.assert_allclose(lse[0], np.log(g["expected_lse_exp"]), rtol=1e-14, atol=1e-14)
    tok, frame, head, aqf = oracle.evidence(q, k, cu, n_vis, g["tokens_per_frame"], scale=1.0)
    np.testing.assert_allclose(tok[0], g["expected_tok"], rtol=1e-13)
    np.testing.assert_allclose(frame[0], g["expected_frame"], rtol=1e-13)
    np.testing.assert_allclose(head[0], g["expected_head"], rtol=1e-13)
    np.testing.assert_allclose(aqf, g["expected_aqf"], rtol=1e-13)


def test_golden_layout_rule():
    # text tiles restart at the text start: n_vis = 5, tile 4 -> visual tiles {0-3} {4}; text {5-8} {9}
    is_text, tid = oracle.token_layout(5, 5, 4)
    assert list(tid) == [0, 0, 0, 0, 1, 2, 2, 2, 2, 3]
    assert list(is_text) == [False] * 5 + [True] * 5


# ---------------------------------------------------------------- O1
def _allowed_count_sink_window(p, n_vis, tile, window):
    """|allowed(p)| for the sink + causal-window mask, counted from tile lengths."""
    if p >= n_vis:
        return p + 1
    r = p // tile
    tiles = ({0} | set(range(max(0, r - window + 1), r))) - {r}
    return sum(min(tile, n_vis - t * tile) for t in tiles) + (p - r * tile + 1)


@pytest.mark.parametrize("window", [1, 2, 3])
def test_O1_constant_keys(window):
    rng = np.random.default_rng(11)
    n_vis, n_text, tile, d = 22, 9, 4, 8          # ragged last visual tile (22 = 5*4 + 2)
    n = n_vis + n_text
    cfg = wl.ProbeConfig("t", (11,), 2, (n_text,), 2, 1, d, tile, window)
    row_ptr, col_idx = wl.build_mask(cfg)
    q = rng.standard_normal((n, 2, d))
    kvec = rng.standard_normal(d)
    k = np.broadcast_to(kvec, (n, 1, d)).copy()
    v = rng.standard_normal((n, 1, d))
    cu = np.array([0, n]); nv = np.array([n_vis])
    scale = 0.37
    o, lse = oracle.probe(q, k, v, cu, nv, tile, row_ptr, col_idx, scale=scale)
    for p in range(n):
        cnt = _allowed_count_sink_window(p, n_vis, tile, window)
        for h in range(2):
            assert abs(lse[h, p] - (scale * q[p, h] @ kvec + math.log(cnt))) < 1e-12
    # O_i is the mean of the allowed values: check against explicit tile arithmetic for a few rows
    p = n_vis - 1                                   # last visual row, ragged tile 5
    r = p // tile
    idx = [j for t in sorted({0} | set(range(max(0, r - window + 1), r + 1)))
           for j in range(t * tile, min((t + 1) * tile, n_vis)) if j <= p]
    np.testing.assert_allclose(o[p, 0], v[idx, 0].mean(axis=0), atol=1e-13)
    np.testing.assert_allclose(o[n - 1, 1], v[:, 0].mean(axis=0), atol=1e-13)
    # evidence with constant keys: P = 1/(p+1) on each text row p
    tok, frame, head, aqf = oracle.evidence(q, k, cu, nv, 2, scale=scale)
    expect = sum(1.0 / (p + 1) for p in range(n_vis, n))
    np.testing.assert_allclose(tok, expect, rtol=1e-13)
    np.testing.assert_allclose(aqf, 2 * expect / n_text, rtol=1e-13)


# ---------------------------------------------------------------- O2
@pytest.mark.parametrize("sharp", [False, True])
def test_O2_row_mass(sharp):
    c = _random_case(2, sharp=sharp)
    hq = c["q"].shape[1]
    for b in range(2):
        nv = int(c["n_vis"][b]); n_text = int(c["cu"][b + 1] - c["cu"][b]) - nv
        for h in range(hq):
            p = oracle.text_probabilities(c["q"], c["k"], c["cu"], c["n_vis"], b, h)
            assert np.all(np.isfinite(p))
            np.testing.assert_allclose(p.sum(axis=1), 1.0, atol=1e-12)
    tok, frame, head, aqf = oracle.evidence(c["q"], c["k"], c["cu"], c["n_vis"], c["npf"])
    for b in range(2):
        nv = int(c["n_vis"][b]); n_text = int(c["cu"][b + 1] - c["cu"][b]) - nv
        for h in range(hq):
            p = oracle.text_probabilities(c["q"], c["k"], c["cu"], c["n_vis"], b, h)
            text_mass = p[:, nv:].sum()
            assert abs(head[b, h] + text_mass - n_text) < 1e-10
    if sharp:
        # large logits: rows must still normalise; LSE finite and above the row max
        o, lse, _ = _run(c)
        assert np.all(np.isfinite(o)) and np.all(np.isfinite(lse))


# ---------------------------------------------------------------- O3
def test_O3_all_tiles_equals_dense_causal_sdpa():
    torch = pytest.importorskip("torch")
    c = _random_case(3, videos=((12, 6), (10, 4)), density=1.0)
    o, lse, _ = _run(c)
    hq, hkv = c["q"].shape[1], c["k"].shape[1]
    for b in range(2):
        s0, s1 = int(c["cu"][b]), int(c["cu"][b + 1])
        qt = torch.from_numpy(c["q"][s0:s1].astype(np.float64)).transpose(0, 1)       # [H, n, d]
        kt = torch.from_numpy(c["k"][s0:s1].astype(np.float64)).transpose(0, 1).repeat_interleave(hq // hkv, 0)
        vt = torch.from_numpy(c["v"][s0:s1].astype(np.float64)).transpose(0, 1).repeat_interleave(hq // hkv, 0)
        ref = torch.nn.functional.scaled_dot_product_attention(qt, kt, vt, is_causal=True)
        np.testing.assert_allclose(o[s0:s1], ref.transpose(0, 1).numpy(), atol=1e-12)


# ---------------------------------------------------------------- O4
def _brute(c, scale):
    """Pure-Python loops straight from the position rules."""
    q, k, v, cu, n_vis, tile = c["q"], c["k"], c["v"], c["cu"], c["n_vis"], c["tile"]
    n, hq, d = q.shape
    hkv = k.shape[1]
    o = [[[0.0] * d for _ in range(hq)] for _ in range(n)]
    lse = [[0.0] * n for _ in range(hq)]
    row = 0
    sets = []
    for b in range(len(n_vis)):
        vs = []
        for _ in range(-(-int(n_vis[b]) // tile)):
            vs.append(set(int(x) for x in c["col_idx"][c["row_ptr"][row]:c["row_ptr"][row + 1]]))
            row += 1
        sets.append(vs)
    for b in range(len(n_vis)):
        s0, s1, nv = int(cu[b]), int(cu[b + 1]), int(n_vis[b])
        for i in range(s0, s1):
            pi = i - s0
            js = []
            for j in range(s0, i + 1):
                pj = j - s0
                if pi >= nv or (pj // tile) in sets[b][pi // tile]:
                    js.append(j)
            for h in range(hq):
                g = h * hkv // hq
                logits = [scale * sum(float(q[i, h, e]) * float(k[j, g, e]) for e in range(d)) for j in js]
                mx = max(logits)
                z = sum(math.exp(x - mx) for x in logits)
                lse[h][i] = mx + math.log(z)
                for e in range(d):
                    o[i][h][e] = sum(math.exp(x - lse[h][i]) * float(v[j, g, e]) for x, j in zip(logits, js))
    return np.array(o), np.array(lse)


@pytest.mark.parametrize("seed,tile,npf", [(4, 4, 2), (5, 8, 4), (6, 4, 4)])
def test_O4_brute_force(seed, tile, npf):
    c = _random_case(seed, videos=((8, 5), (16, 7), (4, 3)), tile=tile, npf=npf, d=6)
    o, lse, (tok, frame, head, aqf) = _run(c)
    scale = 1.0 / math.sqrt(6)
    ob, lb = _brute(c, scale)
    np.testing.assert_allclose(o, ob, atol=1e-12)
    np.testing.assert_allclose(lse, lb, atol=1e-12)
    # evidence by loops: text rows of each video onto its visual tokens
    q, k = c["q"], c["k"]
    hq, hkv = q.shape[1], k.shape[1]
    vis_off = 0
    for b in range(3):
        s0, s1, nv = int(c["cu"][b]), int(c["cu"][b + 1]), int(c["n_vis"][b])
        for h in range(hq):
            g = h * hkv // hq
            for m in range(nv):
                acc = 0.0
                for i in range(s0 + nv, s1):
                    x = scale * sum(float(q[i, h, e]) * float(k[s0 + m, g, e]) for e in range(6))
                    acc += math.exp(x - lb[h][i])
                assert abs(tok[h, vis_off + m] - acc) < 1e-12
        vis_off += nv


# ---------------------------------------------------------------- O5
def test_O5_key_shift_invariance():
    c = _random_case(7)
    o, lse, maps = _run(c)
    shift = np.random.default_rng(1).standard_normal(c["k"].shape[2])
    c2 = dict(c)
    c2["k"] = c["k"].astype(np.float64) + shift               # same shift for every key and KV head
    o2, lse2, maps2 = _run(c2)
    np.testing.assert_allclose(o2, o, atol=1e-12)
    scale = 1.0 / math.sqrt(c["q"].shape[2])
    np.testing.assert_allclose(lse2, lse + scale * (c["q"].astype(np.float64) @ shift).T, atol=1e-12)
    for a, b in zip(maps, maps2):
        np.testing.assert_allclose(a, b, atol=1e-12)


# ---------------------------------------------------------------- O6
def test_O6_gqa_equals_replicated_mha():
    c = _random_case(8, hq=6, hkv=2)
    o, lse, maps = _run(c)
    c2 = dict(c)
    c2["k"] = np.repeat(c["k"], 3, axis=1)          # KV head g serves query heads 3g..3g+2
    c2["v"] = np.repeat(c["v"], 3, axis=1)
    o2, lse2, maps2 = _run(c2)
    np.testing.assert_array_equal(o2, o)
    np.testing.assert_array_equal(lse2, lse)
    for a, b in zip(maps, maps2):
        np.testing.assert_array_equal(a, b)


# ---------------------------------------------------------------- O7
def test_O7_varlen_independence():
    c = _random_case(9, videos=((8, 3), (12, 6), (4, 2)))
    o, lse, (tok, frame, head, aqf) = _run(c)
    row = 0
    vis0 = fr0 = 0
    for b in range(3):
        s0, s1, nv = int(c["cu"][b]), int(c["cu"][b + 1]), int(c["n_vis"][b])
        nvt = -(-nv // c["tile"])
        rp = c["row_ptr"][row:row + nvt + 1] - c["row_ptr"][row]
        ci = c["col_idx"][c["row_ptr"][row]:c["row_ptr"][row + nvt]]
        row += nvt
        one = dict(q=c["q"][s0:s1], k=c["k"][s0:s1], v=c["v"][s0:s1], cu=np.array([0, s1 - s0]),
                   n_vis=np.array([nv]), tile=c["tile"], npf=c["npf"], row_ptr=rp, col_idx=ci)
        ob, lb, (tb, fb, hb, ab) = _run(one)
        np.testing.assert_array_equal(ob, o[s0:s1])
        np.testing.assert_array_equal(lb, lse[:, s0:s1])
        nf = nv // c["npf"]
        np.testing.assert_array_equal(tb, tok[:, vis0:vis0 + nv])
        np.testing.assert_array_equal(fb, frame[:, fr0:fr0 + nf])
        np.testing.assert_array_equal(hb[0], head[b])
        np.testing.assert_array_equal(ab, aqf[fr0:fr0 + nf])
        vis0 += nv; fr0 += nf


# ---------------------------------------------------------------- O8
def test_O8_reductions():
    c = _random_case(10, videos=((8, 3), (12, 6)), npf=4)
    tok, frame, head, aqf = oracle.evidence(c["q"], c["k"], c["cu"], c["n_vis"], 4)
    hq = c["q"].shape[1]
    vis0 = fr0 = 0
    for b in range(2):
        nv = int(c["n_vis"][b]); nf = nv // 4
        n_text = int(c["cu"][b + 1] - c["cu"][b]) - nv
        for t in range(nf):
            for h in range(hq):
                assert abs(frame[h, fr0 + t] - sum(tok[h, vis0 + 4 * t + u] for u in range(4))) < 1e-14
            assert abs(aqf[fr0 + t] - sum(frame[h, fr0 + t] for h in range(hq)) / (hq * n_text)) < 1e-14
        for h in range(hq):
            assert abs(head[b, h] - frame[h, fr0:fr0 + nf].sum()) < 1e-13
        assert aqf[fr0:fr0 + nf].sum() <= 1.0 + 1e-12
        assert np.all(tok[:, vis0:vis0 + nv] >= 0)
        vis0 += nv; fr0 += nf


# ---------------------------------------------------------------- O9
@pytest.mark.parametrize("name", ["tiny", "single"])
def test_O9_planted_frames_rank_top(name):
    p = wl.make_probe(wl.CONFIGS[name])
    tok, frame, head, aqf = oracle.evidence(p.q, p.k, p.cu_seqlens, p.n_vis, p.cfg.tokens_per_frame)
    planted = p.planted[0]
    top = np.sort(np.argsort(-frame.sum(axis=0), kind="stable")[:planted.size])
    np.testing.assert_array_equal(top, planted)
    top_aqf = np.sort(np.argsort(-aqf, kind="stable")[:planted.size])
    np.testing.assert_array_equal(top_aqf, planted)


# ---------------------------------------------------------------- O10
def test_O10_linearity_in_v():
    c = _random_case(12)
    rng = np.random.default_rng(5)
    v2 = rng.standard_normal(c["v"].shape)
    o1, _, _ = _run(c)
    c2 = dict(c); c2["v"] = v2
    o2, _, _ = _run(c2)
    c3 = dict(c); c3["v"] = 2.5 * c["v"].astype(np.float64) - 0.75 * v2
    o3, _, _ = _run(c3)
    np.testing.assert_allclose(o3, 2.5 * o1 - 0.75 * o2, atol=1e-12)


# ---------------------------------------------------------------- planted mistakes
def test_pins_catch_planted_mistakes(monkeypatch):
    """A wrong mask rule or a wrong GQA grouping in the oracle must fail a pin."""
    import oracle.attention as op
    g = json.load(open(os.path.join(GOLDEN, "hand_mask_example.json")))
    n = len(g["q"])
    q = np.ones((n, 1, 1)); k = np.log(np.array(g["k_exp"], float)).reshape(n, 1, 1)
    v = np.array(g["v"], float).reshape(n, 1, 1)
    good = op.allowed_row

    def ignores_mask(p, is_text, tile_id, retained):       # planted mistake: dense causal rows
        return good(p, np.ones_like(is_text), tile_id, retained)
    monkeypatch.setattr(op, "allowed_row", ignores_mask)
    o, _ = op.probe(q, k, v, np.array([0, n]), np.array([4]), 2, np.array(g["row_ptr"]),
                    np.array(g["col_idx"]), scale=1.0)
    assert not np.allclose(o[:, 0, 0], g["expected_o"])


# ---------------------------------------------------------------- intra-frame cue A_if
# Pins of oracle.intra_frame (Sec. 3.2, "Evidence Decomposition"):
#   F1  closed form for constant keys: P = 1/|allowed(row)| on j <= i
#   F2  all-tiles mask: the diagonal frame blocks of dense causal attention
#       weights (torch softmax over masked logits, float64), head-averaged
#   F3  brute force, pure-Python loops, random masks, varlen
#   F4  structure: zero above the diagonal; a video's first frame is
#       row-stochastic (its rows see only their own frame); rows sum to <= 1
def test_F1_intra_frame_constant_keys():
    rng = np.random.default_rng(21)
    n_vis, n_text, tile, d, npf, window = 24, 5, 8, 8, 4, 2
    n = n_vis + n_text
    cfg = wl.ProbeConfig("t", (n_vis // npf,), npf, (n_text,), 2, 1, d, tile, window)
    row_ptr, col_idx = wl.build_mask(cfg)
    q = rng.standard_normal((n, 2, d))
    k = np.broadcast_to(rng.standard_normal(d), (n, 1, d)).copy()
    a = oracle.intra_frame(q, k, [0, n], [n_vis], npf, tile, row_ptr, col_idx, scale=0.3)
    for t in range(n_vis // npf):
        for i in range(npf):
            p = t * npf + i
            cnt = _allowed_count_sink_window(p, n_vis, tile, window)
            for j in range(npf):
                want = 1.0 / cnt if j <= i else 0.0
                assert abs(a[t, i, j] - want) < 1e-13, (t, i, j)


def test_F2_intra_frame_all_tiles_equals_dense_causal_weights():
    torch = pytest.importorskip("torch")
    c = _random_case(23, videos=((12, 6), (8, 4)), density=1.0, tile=4, npf=4)
    a = oracle.intra_frame(c["q"], c["k"], c["cu"], c["n_vis"], 4, c["tile"], c["row_ptr"], c["col_idx"])
    hq, hkv, d = c["q"].shape[1], c["k"].shape[1], c["q"].shape[2]
    f = 0
    for b in range(2):
        s0, s1, nv = int(c["cu"][b]), int(c["cu"][b + 1]), int(c["n_vis"][b])
        qt = torch.from_numpy(c["q"][s0:s1].astype(np.float64)).transpose(0, 1)
        kt = torch.from_numpy(c["k"][s0:s1].astype(np.float64)).transpose(0, 1).repeat_interleave(hq // hkv, 0)
        logits = qt @ kt.transpose(1, 2) / math.sqrt(d)
        n = s1 - s0
        logits = logits.masked_fill(torch.triu(torch.ones(n, n, dtype=torch.bool), 1), float("-inf"))
        w = torch.softmax(logits, dim=-1).mean(dim=0).numpy()        # head-averaged weights
        for t in range(nv // 4):
            np.testing.assert_allclose(a[f], w[4 * t:4 * t + 4, 4 * t:4 * t + 4], atol=1e-13)
            f += 1


@pytest.mark.parametrize("seed,tile,npf", [(24, 4, 2), (25, 8, 4)])
def test_F3_intra_frame_brute_force(seed, tile, npf):
    c = _random_case(seed, videos=((8, 3), (16, 5)), tile=tile, npf=npf, d=5)
    a = oracle.intra_frame(c["q"], c["k"], c["cu"], c["n_vis"], npf, tile, c["row_ptr"], c["col_idx"])
    _, lb = _brute(c, 1.0 / math.sqrt(5))
    q, k = c["q"], c["k"]
    hq, hkv = q.shape[1], k.shape[1]
    f = 0
    for b in range(2):
        s0, nv = int(c["cu"][b]), int(c["n_vis"][b])
        for t in range(nv // npf):
            for i in range(npf):
                row = s0 + t * npf + i
                for j in range(npf):
                    key = s0 + t * npf + j
                    acc = 0.0
                    if j <= i:     # the diagonal tile is always kept
                        for h in range(hq):
                            x = sum(float(q[row, h, e]) * float(k[key, h * hkv // hq, e]) for e in range(5))
                            acc += math.exp(x / math.sqrt(5) - lb[h][row]) / hq
                    assert abs(a[f, i, j] - acc) < 1e-12
            f += 1


def test_F4_intra_frame_structure():
    c = _random_case(26, videos=((16, 4), (12, 5)), tile=8, npf=4, sharp=True)
    a = oracle.intra_frame(c["q"], c["k"], c["cu"], c["n_vis"], 4, c["tile"], c["row_ptr"], c["col_idx"])
    assert np.all(np.triu(a, 1) == 0.0)
    assert np.all(a.sum(axis=2) <= 1.0 + 1e-12)
    np.testing.assert_allclose(a[0].sum(axis=1), 1.0, atol=1e-12)          # video 0, frame 0
    np.testing.assert_allclose(a[4].sum(axis=1), 1.0, atol=1e-12)          # video 1, frame 0
    # a frame selection returns the same rows
    sel = oracle.intra_frame(c["q"], c["k"], c["cu"], c["n_vis"], 4, c["tile"], c["row_ptr"], c["col_idx"],
                             frames=[6, 1])
    np.testing.assert_array_equal(sel, a[[6, 1]])


def test_F1_catches_a_frame_local_softmax(monkeypatch):
    """Planted mistake: normalising inside the frame instead of over the row's allowed keys."""
    import oracle.attention as op
    good = op._attend
    npf = 4                                            # the frame size test_F1 uses

    def frame_local(qh, kh, vh, allowed, scale):
        o, lse, p = good(qh, kh, vh, allowed, scale)
        out = np.zeros_like(p)
        for r in range(p.shape[0]):
            f0 = (np.nonzero(p[r])[0].max() // npf) * npf   # the row's own frame (its last allowed key is itself)
            out[r, f0:f0 + npf] = p[r, f0:f0 + npf] / p[r, f0:f0 + npf].sum()
        return o, lse, out
    monkeypatch.setattr(op, "_attend", frame_local)
    with pytest.raises(AssertionError):
        test_F1_intra_frame_constant_keys()


# ---------------------------------------------------------------- cross-frame cue A_ff, E_ff
# Pins of oracle.frame_mass_rows / cross_frame / e_ff (Sec. 3.2, "Evidence
# Decomposition"):
#   G1  closed form for constant keys: A_ff[a-1, b] = mean over a's rows of
#       |allowed(i) within frame b| / |allowed(i)|, counted from the tile rules
#   G2  mass balance with the separately pinned A_if: for every frame,
#       sum_b A_ff[a-1, b] + (1/N_v) sum_ij A_if[a, i, j] = 1 (a row's
#       probabilities over its earlier frames and its own frame sum to one)
#   G3  brute force, pure-Python loops, random masks, varlen
#   G4  all-tiles mask: frame-block means of dense causal attention weights
#       (torch softmax over masked logits, float64), head-averaged
#   G5  E_ff on a hand-worked 3-frame example
def test_G1_cross_frame_constant_keys():
    rng = np.random.default_rng(31)
    n_vis, n_text, tile, d, npf, window = 32, 5, 8, 8, 4, 2
    n = n_vis + n_text
    cfg = wl.ProbeConfig("t", (n_vis // npf,), npf, (n_text,), 2, 1, d, tile, window)
    row_ptr, col_idx = wl.build_mask(cfg)
    q = rng.standard_normal((n, 2, d))
    k = np.broadcast_to(rng.standard_normal(d), (n, 1, d)).copy()
    aff, _ = oracle.cross_frame(q, k, [0, n], [n_vis], npf, tile, row_ptr, col_idx, scale=0.3)
    T = n_vis // npf
    assert aff[0].shape == (T - 1, T - 1)
    for a in range(1, T):
        for b in range(T - 1):
            want = 0.0
            if b < a:
                for i in range(npf):
                    p = a * npf + i
                    r = p // tile
                    kept = {0} | set(range(max(0, r - window + 1), r + 1))
                    inside = npf if (b * npf) // tile in kept else 0      # frame b lies in one tile, before row p
                    want += inside / _allowed_count_sink_window(p, n_vis, tile, window) / npf
            assert abs(aff[0][a - 1, b] - want) < 1e-13, (a, b)


def test_G2_cross_frame_mass_balance():
    c = _random_case(32, videos=((24, 5), (16, 7), (4, 3)), tile=8, npf=4, sharp=True)
    args = (c["q"], c["k"], c["cu"], c["n_vis"], 4, c["tile"], c["row_ptr"], c["col_idx"])
    aff, eff = oracle.cross_frame(*args)
    aif = oracle.intra_frame(*args)
    f = 0
    for b, nv in enumerate(c["n_vis"]):
        T = int(nv) // 4
        for a in range(T):
            earlier = aff[b][a - 1, :a].sum() if a >= 1 else 0.0
            assert abs(earlier + aif[f].sum() / 4 - 1.0) < 1e-12, (b, a)
            f += 1
    assert eff.shape == (f,)
    # the rows a frame selection returns are those of the full cue
    rows = oracle.frame_mass_rows(*args, frames=[3, 7])
    np.testing.assert_allclose(rows[0][:3], aff[0][2, :3], atol=0)
    np.testing.assert_allclose(rows[1][:1], aff[1][0, :1], atol=0)


@pytest.mark.parametrize("seed,tile,npf", [(33, 4, 2), (34, 8, 4)])
def test_G3_cross_frame_brute_force(seed, tile, npf):
    c = _random_case(seed, videos=((12, 3), (16, 5)), tile=tile, npf=npf, d=5)
    aff, eff = oracle.cross_frame(c["q"], c["k"], c["cu"], c["n_vis"], npf, tile, c["row_ptr"], c["col_idx"])
    _, lb = _brute(c, 1.0 / math.sqrt(5))
    q, k, cu, n_vis = c["q"], c["k"], c["cu"], c["n_vis"]
    hq, hkv = q.shape[1], k.shape[1]
    row = 0
    for b in range(2):
        s0, nv = int(cu[b]), int(n_vis[b])
        kept = []
        for _ in range(-(-nv // tile)):
            kept.append(set(int(x) for x in c["col_idx"][c["row_ptr"][row]:c["row_ptr"][row + 1]]))
            row += 1
        T = nv // npf
        for a in range(1, T):
            for fb in range(a):
                acc = 0.0
                for i in range(npf):
                    pi = a * npf + i
                    for j in range(npf):
                        pj = fb * npf + j
                        if pj // tile not in kept[pi // tile]:
                            continue
                        for h in range(hq):
                            x = sum(float(q[s0 + pi, h, e]) * float(k[s0 + pj, h * hkv // hq, e]) for e in range(5))
                            acc += math.exp(x / math.sqrt(5) - lb[h][s0 + pi]) / (npf * hq)
                assert abs(aff[b][a - 1, fb] - acc) < 1e-12, (b, a, fb)
            for fb in range(a, T - 1):
                assert aff[b][a - 1, fb] == 0.0


def test_G4_cross_frame_all_tiles_equals_dense_causal_weights():
    torch = pytest.importorskip("torch")
    c = _random_case(35, videos=((16, 6), (12, 4)), density=1.0, tile=4, npf=4)
    aff, _ = oracle.cross_frame(c["q"], c["k"], c["cu"], c["n_vis"], 4, c["tile"], c["row_ptr"], c["col_idx"])
    hq, hkv, d = c["q"].shape[1], c["k"].shape[1], c["q"].shape[2]
    for b in range(2):
        s0, s1, nv = int(c["cu"][b]), int(c["cu"][b + 1]), int(c["n_vis"][b])
        qt = torch.from_numpy(c["q"][s0:s1].astype(np.float64)).transpose(0, 1)
        kt = torch.from_numpy(c["k"][s0:s1].astype(np.float64)).transpose(0, 1).repeat_interleave(hq // hkv, 0)
        logits = qt @ kt.transpose(1, 2) / math.sqrt(d)
        n = s1 - s0
        logits = logits.masked_fill(torch.triu(torch.ones(n, n, dtype=torch.bool), 1), float("-inf"))
        w = torch.softmax(logits, dim=-1).mean(dim=0).numpy()
        T = nv // 4
        blocks = w[:nv, :nv].reshape(T, 4, T, 4).sum(axis=3).mean(axis=1)      # [a, b]: mean row mass
        np.testing.assert_allclose(aff[b], np.tril(blocks[1:, :T - 1]), atol=1e-13)


def test_G5_e_ff_hand_example():
    # frames 0, 1, 2: A(1->0) = 0.2, A(2->0) = 0.3, A(2->1) = 0.4
    aff = [np.array([[0.2, 0.0], [0.3, 0.4]])]
    e = oracle.e_ff(aff, [3])
    # E[0] = (0 + 0.2 + 0.3)/2, E[1] = (0.2 + 0.4)/2, E[2] = (0.3 + 0.4 + 0)/2
    np.testing.assert_allclose(e, [0.25, 0.30, 0.35], atol=1e-15)
    np.testing.assert_array_equal(oracle.e_ff([np.zeros((0, 0))], [1]), [0.0])


def test_G5_catches_a_shifted_receive_column(monkeypatch):
    """Planted mistake: the received attention read from column t - 1."""
    import oracle.attention as op

    def shifted(aff, n_frames):
        out = []
        for a_b, tb in zip(aff, n_frames):
            e = np.zeros(int(tb))
            for t in range(int(tb)):
                give = a_b[t - 1, :t].sum() if t >= 1 else 0.0
                recv = a_b[t:, t - 1].sum() if 1 <= t <= tb - 2 else 0.0
                e[t] = 0.5 * (give + recv)
            out.append(e)
        return np.concatenate(out)
    monkeypatch.setattr(op, "e_ff", shifted)
    monkeypatch.setattr(oracle, "e_ff", shifted)
    with pytest.raises(AssertionError):
        test_G5_e_ff_hand_example()


def test_G1_catches_a_block_mean_over_all_pairs(monkeypatch):
    """Planted mistake: A_ff as the mean over all N_v x N_v entries (an extra 1/N_v)."""
    import oracle.attention as op
    good = op.frame_mass_rows

    def per_entry(*a, **kw):
        return [r / 4 for r in good(*a, **kw)]                 # N_v = 4 in test_G1
    monkeypatch.setattr(op, "frame_mass_rows", per_entry)
    with pytest.raises(AssertionError):
        test_G1_cross_frame_constant_keys()


# ---------------------------------------------------------------- top-p block retention (Eq. 6-9)
# Pins of oracle.topp:
#   H1  constant keys: uniform p over H_i, so S_i is the ceil(tau |H_i|)
#       lowest block ids (the tie rule), counted without any softmax
#   H2  brute force, pure-Python block means, logits, softmax and sort
#   H3  a planted block aligned with the row's query takes all the mass
#   H4  monotone in tau; tau -> 1 keeps all of H_i; tiny tau keeps the argmax
#   H5  keeping every block equals dense causal attention (torch, float64)
def _topp_case(seed, videos=((32, 9), (24, 5)), hq=4, hkv=2, d=8, block=4):
    rng = np.random.default_rng(seed)
    n_vis = np.array([a for a, _ in videos], np.int32)
    lens = np.array([a + b for a, b in videos])
    cu = np.concatenate([[0], np.cumsum(lens)]).astype(np.int32)
    n = int(cu[-1])
    q = wl.bf16_round(rng.standard_normal((n, hq, d)).astype(np.float32))
    k = wl.bf16_round(rng.standard_normal((n, hkv, d)).astype(np.float32))
    v = wl.bf16_round(rng.standard_normal((n, hkv, d)).astype(np.float32))
    return dict(q=q, k=k, v=v, cu=cu, n_vis=n_vis, block=block)


def test_H1_topp_constant_keys():
    c = _topp_case(41)
    k = np.broadcast_to(c["k"][0:1], c["k"].shape).copy()
    tau = 0.93          # tau * n stays away from integers for n <= 15 (no cumulative-sum rounding ties)
    sets, probs = oracle.retained_blocks(c["q"], k, c["cu"], c["n_vis"], 4, tau)
    for b in range(2):
        s0, s1, nv = int(c["cu"][b]), int(c["cu"][b + 1]), int(c["n_vis"][b])
        nb = nv // 4 + -(-(s1 - s0 - nv) // 4)
        for row in range(s0, s1):
            # blocks ending before the row: every block whose start + length <= local position
            n_hist = sum(1 for s, ln in oracle.block_layout(nv, s1 - s0 - nv, 4) if s + ln <= row - s0)
            assert n_hist <= nb
            want = list(range(math.ceil(tau * n_hist))) if n_hist else []
            for h in range(4):
                assert sets[(h, row)] == want, (b, row, h)


@pytest.mark.parametrize("seed", [42, 43])
def test_H2_topp_brute_force(seed):
    c = _topp_case(seed, videos=((16, 7), (12, 3)), d=5, block=4)
    tau = 0.8
    sets, _ = oracle.retained_blocks(c["q"], c["k"], c["cu"], c["n_vis"], 4, tau)
    q, k = c["q"], c["k"]
    hq, hkv = q.shape[1], k.shape[1]
    for b in range(2):
        s0, s1, nv = int(c["cu"][b]), int(c["cu"][b + 1]), int(c["n_vis"][b])
        blocks = [(s, 4) for s in range(0, nv, 4)] + [(nv + s, min(4, s1 - s0 - nv - s)) for s in range(0, s1 - s0 - nv, 4)]
        for row in range(s0, s1):
            for h in range(hq):
                g = []
                for j, (s, ln) in enumerate(blocks):
                    if s + ln > row - s0:
                        continue
                    kb = [sum(float(k[s0 + s + t, h * hkv // hq, e]) for t in range(ln)) / ln for e in range(5)]
                    g.append((j, sum(float(q[row, h, e]) * kb[e] for e in range(5)) / math.sqrt(5)))
                if not g:
                    assert sets[(h, row)] == []
                    continue
                mx = max(x for _, x in g)
                z = sum(math.exp(x - mx) for _, x in g)
                ranked = sorted(((-math.exp(x - mx) / z, j) for j, x in g))
                acc, keep = 0.0, []
                for negp, j in ranked:
                    if acc >= tau:
                        break
                    keep.append(j)
                    acc += -negp
                assert sets[(h, row)] == sorted(keep), (b, row, h)


def test_H3_topp_planted_block_takes_the_mass():
    c = _topp_case(44, videos=((32, 6),), hq=2, hkv=2)
    q, k = c["q"], c["k"].copy()
    row = 35                                          # a text row; block 3 (tokens 12..15) is planted
    for h in range(2):
        k[12:16, h, :] = 40.0 * q[row, h, :] / np.linalg.norm(q[row, h, :])
    sets, probs = oracle.retained_blocks(q, k, c["cu"], c["n_vis"], 4, 0.97, rows=[row])
    for h in range(2):
        assert sets[(h, row)] == [3], h


def test_H4_topp_monotone_and_limits():
    c = _topp_case(45)
    args = (c["q"], c["k"], c["cu"], c["n_vis"], 4)
    rows = [10, 20, 33, 40, 55, 60]
    s_lo, _ = oracle.retained_blocks(*args, 0.5, rows=rows)
    s_hi, probs = oracle.retained_blocks(*args, 0.95, rows=rows)
    s_all, _ = oracle.retained_blocks(*args, 1.0 - 1e-12, rows=rows)
    s_one, _ = oracle.retained_blocks(*args, 1e-9, rows=rows)
    for key in s_lo:
        hist, p = probs[key]
        assert set(s_lo[key]) <= set(s_hi[key]) <= set(s_all[key])
        assert s_all[key] == [int(j) for j in hist]
        assert s_one[key] == ([int(hist[np.argmax(p)])] if hist.size else [])
        if hist.size:
            kept = np.isin(hist, s_hi[key])
            assert p[kept].sum() >= 0.95 - 1e-12
            assert p[kept].sum() - p[kept].min() < 0.95            # minimal
            assert p[kept].min() >= p[~kept].max(initial=0.0)       # a top set


def test_H5_topp_keep_all_equals_dense_causal():
    torch = pytest.importorskip("torch")
    c = _topp_case(46, videos=((16, 5),))
    rows = np.arange(21)
    sets, probs = oracle.retained_blocks(c["q"], c["k"], c["cu"], c["n_vis"], 4, 1.0 - 1e-12, rows=rows)
    o, lse = oracle.probe_rows_topp(c["q"], c["k"], c["v"], c["cu"], c["n_vis"], 4, sets, rows)
    qt = torch.from_numpy(c["q"].astype(np.float64)).transpose(0, 1)
    kt = torch.from_numpy(c["k"].astype(np.float64)).transpose(0, 1).repeat_interleave(2, 0)
    vt = torch.from_numpy(c["v"].astype(np.float64)).transpose(0, 1).repeat_interleave(2, 0)
    ref = torch.nn.functional.scaled_dot_product_attention(qt, kt, vt, is_causal=True).transpose(0, 1).numpy()
    np.testing.assert_allclose(o, ref, atol=1e-12)


def test_H3_catches_an_ascending_order(monkeypatch):
    """Planted mistake: ranking H_i by p ascending."""
    import oracle.topp as ot

    def ascending(p, tau):
        order = sorted(range(len(p)), key=lambda j: (p[j], j))
        acc, keep = 0.0, []
        for j in order:
            if acc >= tau:
                break
            keep.append(j)
            acc += p[j]
        return sorted(keep)
    monkeypatch.setattr(ot, "select_prefix", ascending)
    with pytest.raises(AssertionError):
        test_H3_topp_planted_block_takes_the_mass()


def test_H7_evidence_with_every_block_kept_is_the_dense_evidence():
    c = _topp_case(48, videos=((16, 6), (12, 5)))
    sets, _ = oracle.retained_blocks(c["q"], c["k"], c["cu"], c["n_vis"], 4, 1.0 - 1e-12)
    got = oracle.evidence_topp(c["q"], c["k"], c["cu"], c["n_vis"], 4, 4, sets)
    want = oracle.evidence(c["q"], c["k"], c["cu"], c["n_vis"], 4)
    for g, w in zip(got, want):
        np.testing.assert_allclose(g, w, atol=1e-13)


# Pins of oracle.topp.coarse_evidence (Appendix Eq. 10-11):
#   C1  blocks of one token: g is the exact logit, so the coarse map is the
#       exact attention on the same retained sets (evidence_topp)
#   C2  constant keys: a block's mean is its keys, so again the exact map
#   C3  mass: each text row's coarse map sums to 1, so the token map plus the
#       rows' own-block mass is n_text per head
def test_C1_coarse_with_one_token_blocks_is_exact():
    c = _topp_case(51, videos=((12, 5), (8, 4)))
    sets, _ = oracle.retained_blocks(c["q"], c["k"], c["cu"], c["n_vis"], 1, 0.8)
    got = oracle.coarse_evidence(c["q"], c["k"], c["cu"], c["n_vis"], 4, 1, sets)
    want = oracle.evidence_topp(c["q"], c["k"], c["cu"], c["n_vis"], 4, 1, sets)
    for g, w in zip(got, want):
        np.testing.assert_allclose(g, w, atol=1e-13)


def test_C2_coarse_with_constant_keys_is_exact():
    c = _topp_case(52, videos=((16, 6),))
    k = np.broadcast_to(c["k"][0:1], c["k"].shape).copy()
    sets, _ = oracle.retained_blocks(c["q"], k, c["cu"], c["n_vis"], 4, 0.7)
    got = oracle.coarse_evidence(c["q"], k, c["cu"], c["n_vis"], 4, 4, sets)
    want = oracle.evidence_topp(c["q"], k, c["cu"], c["n_vis"], 4, 4, sets)
    for g, w in zip(got, want):
        np.testing.assert_allclose(g, w, atol=1e-13)


def test_C3_coarse_mass():
    c = _topp_case(53, videos=((16, 6),), hq=2, hkv=1)
    sets, _ = oracle.retained_blocks(c["q"], c["k"], c["cu"], c["n_vis"], 4, 0.9)
    tok, frame, head, aqf = oracle.coarse_evidence(c["q"], c["k"], c["cu"], c["n_vis"], 4, 4, sets)
    # rows 16..21 are text; their own text block (16..19 or 20..21) holds the rest of the mass
    q, k = c["q"].astype(np.float64), c["k"].astype(np.float64)
    for h in range(2):
        rest = 0.0
        for row in range(16, 22):
            so = 16 if row < 20 else 20
            kb = oracle.block_means(c["k"], 16, 6, 4)
            a = {}
            for j in sets[(h, row)]:
                s, ln = oracle.block_layout(16, 6, 4)[j]
                for m in range(s, s + ln):
                    a[m] = float(kb[j, 0] @ q[row, h]) / math.sqrt(8)
            for m in range(so, row + 1):
                a[m] = float(k[m, 0] @ q[row, h]) / math.sqrt(8)
            mx = max(a.values())
            z = sum(math.exp(v - mx) for v in a.values())
            rest += sum(math.exp(v - mx) for m, v in a.items() if m >= 16) / z
        assert abs(tok[h].sum() + rest - 6.0) < 1e-12


def test_C2_catches_block_sums_for_means(monkeypatch):
    """Planted mistake: k_bar as the sum of the block's keys instead of their mean."""
    import oracle.topp as ot
    good = ot.block_means

    def sums(k_video, n_vis, n_text, block):
        m = good(k_video, n_vis, n_text, block)
        lens = np.array([ln for _, ln in ot.block_layout(n_vis, n_text, block)], np.float64)
        return m * lens[:, None, None]
    monkeypatch.setattr(ot, "block_means", sums)
    with pytest.raises(AssertionError):
        test_C2_coarse_with_constant_keys_is_exact()
