"""A synthetic analogue of the paper's sparse-vs-dense comparison (Appendix,
"Detailed Sparse Prefilling": the evidence under top-p block retention should
rank frames as the dense evidence does). A regression signal, not parity: the
oracle's A_qf under the top-p sets (exact logits on retained blocks, and the
Eq. 10-11 coarse map) against the dense-causal A_qf, by Pearson correlation
and top-10% frame overlap, on inputs whose logits have unit scale (N(0, 1)
entries without the extra 1/sqrt(d), so attention is neither uniform nor
one-hot) and a few planted query-aligned frames carry the evidence."""
import numpy as np
import pytest

import oracle
from paper_2608_05780_gb300 import workloads as wl


def _agreement(a, b):
    r = float(np.corrcoef(a, b)[0, 1])
    k = max(1, int(round(0.1 * len(a))))
    top_a = set(np.argsort(-a, kind="stable")[:k])
    top_b = set(np.argsort(-b, kind="stable")[:k])
    return r, len(top_a & top_b) / k


@pytest.mark.parametrize("tau", [0.9, 0.97])
def test_topp_and_coarse_evidence_track_the_dense_evidence(tau):
    # 64 frames x 16 tokens + 48 text rows, 5 planted (query-aligned) frames
    cfg = wl.ProbeConfig("signal", (64,), 16, (48,), 4, 2, 64, 64, 2, plant=(5,), seed=11, mask_seed=11,
                         scale_inputs=False)
    p = wl.make_probe(cfg)
    dense = oracle.evidence(p.q, p.k, p.cu_seqlens, p.n_vis, 16)
    rows = np.arange(int(p.n_vis[0]), int(p.cu_seqlens[-1]))     # the text rows drive the evidence
    sets, _ = oracle.retained_blocks(p.q, p.k, p.cu_seqlens, p.n_vis, 16, tau, rows=rows)
    sparse = oracle.evidence_topp(p.q, p.k, p.cu_seqlens, p.n_vis, 16, 16, sets)
    coarse = oracle.coarse_evidence(p.q, p.k, p.cu_seqlens, p.n_vis, 16, 16, sets)
    planted = set(int(f) for f in p.planted[0])
    assert planted <= set(np.argsort(-dense[3], kind="stable")[:len(planted) + 1].tolist())
    r_s, ov_s = _agreement(dense[3], sparse[3])
    r_c, ov_c = _agreement(dense[3], coarse[3])
    assert r_s > 0.97 and ov_s >= 0.8, (r_s, ov_s)
    assert r_c > 0.9 and ov_c >= 0.8, (r_c, ov_c)
