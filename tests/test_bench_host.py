"""bench.py's mirror of the work planner's text-row split rule (CPU only).

The planner cuts each text row tile's kv list into ranges of
max(longest visual row, 8, min(64, tile work / SMs / 2)) tiles; the bench uses
the same rule to tell whether the probe call launches the split-KV combine,
which its gpu_launches count depends on."""
import os
import sys

import numpy as np
import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

import bench  # noqa: E402
from paper_2608_05780_gb300 import workloads as wl  # noqa: E402


def _split_len(probe, sms):
    """The rule written out from its statement, for the check below."""
    cfg = probe.cfg
    counts = np.diff(probe.row_ptr)
    blocks = cfg.hkv * -(-(cfg.hq // cfg.hkv) // (2 * (128 // cfg.tile)))
    text_rows = [-(-int(nv) // cfg.tile) + t + 1
                 for nv, nt in zip(probe.n_vis, probe.n_text) for t in range(-(-int(nt) // cfg.tile))]
    work = (int(counts.sum()) + sum(text_rows)) * blocks
    return max(int(counts.max()), 8, min(64, work // sms // 2)), text_rows


@pytest.mark.parametrize("name,want_len", [("tiny", 8), ("single", 9), ("long65k", 64)])
def test_split_length_and_combine(name, want_len):
    probe = wl.make_probe(wl.CONFIGS[name])
    split, text_rows = _split_len(probe, 152)
    assert split == want_len
    assert bench._has_combine(probe, 152) == any(r > split for r in text_rows)
    assert bench._has_combine(probe, 152)          # every workload's text row is split


def test_short_text_row_needs_no_combine():
    # 4 frames x 16 tokens (one 64-token tile) + 16 text tokens: the text row
    # attends to 2 tiles, fewer than the minimum range of 8.
    cfg = wl.ProbeConfig("t", (4,), 16, (16,), 2, 1, 64, 64, 2, plant=(1,), seed=3,
                         description="tiny single-tile probe")
    probe = wl.make_probe(cfg)
    assert not bench._has_combine(probe, 152)
