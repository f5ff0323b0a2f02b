"""Seeded input generator: shapes, mask structure, counts (CPU only)."""
import numpy as np
import pytest

from paper_2608_05780_gb300 import workloads as wl


@pytest.mark.parametrize("name,kept", [("tiny", 30), ("single", 183), ("depth28", 1245),
                                       ("long65k", 24425), ("varlen8", 17843)])
def test_kept_tile_counts(name, kept):
    cfg = wl.CONFIGS[name]
    row_ptr, col_idx = wl.build_mask(cfg)
    text = 0
    for nv, nt in zip(cfg.n_vis, cfg.n_text):
        a, b = wl.video_tiles(nv, nt, cfg.tile)
        text += sum(a + t + 1 for t in range(b))
    assert len(col_idx) + text == kept
    # every row sorted, causal, with sink and diagonal
    r = 0
    for nv in cfg.n_vis:
        for t in range(-(-nv // cfg.tile)):
            row = col_idx[row_ptr[r]:row_ptr[r + 1]]
            assert np.all(np.diff(row) > 0) and row[0] == 0 and row[-1] == t
            r += 1


def test_varlen_lengths():
    cfg = wl.CONFIGS["varlen8"]
    assert cfg.frames == (1628, 1961, 1866, 1297, 1957, 2012, 2003, 636)
    assert cfg.n_text == (151, 181, 118, 136, 185, 218, 176, 97)
    assert cfg.n_tot == 215022


def test_bf16_round_matches_torch():
    torch = pytest.importorskip("torch")
    x = (np.random.default_rng(0).standard_normal(100000) * 7).astype(np.float32)
    ref = torch.from_numpy(x).to(torch.bfloat16).float().numpy()
    np.testing.assert_array_equal(wl.bf16_round(x), ref)


def test_tiny_probe_inputs():
    p = wl.make_probe(wl.CONFIGS["tiny"])
    assert p.q.shape == (544, 4, 64) and p.k.shape == (544, 2, 64)
    assert list(p.cu_seqlens) == [0, 544] and list(p.n_vis) == [512]
    assert np.array_equal(wl.bf16_round(p.q), p.q)
    assert len(p.planted[0]) == 3
    again = wl.make_probe(wl.CONFIGS["tiny"])
    assert np.array_equal(p.k, again.k)
