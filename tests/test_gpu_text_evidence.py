"""GPU parity of the recompute evidence pass (evisel_probe_args.text_evidence = 1):
the token / frame / head maps and A_qf formed from q and k and the probe's
LSE, with no text-row logit spill, against the float64 oracle on the seeded
workloads and edge cases, against the spill path on the same inputs, summed
over layers, and through the entry point that allocates nothing (the 65K
probe fits its 64 MiB scratch without the spill).

Tolerances are those of the spill path (frame evidence <= 1e-3 abs per entry
after dividing by the text-row count, identical top-k planted frames); the
two paths differ only in fp32 summation order and in the logits (bf16 MMA
products accumulated in fp32 in both), so they agree to about 1e-5 relative.
"""
import numpy as np
import pytest

import oracle
from paper_2608_05780_gb300 import _binding as B
from paper_2608_05780_gb300 import workloads as wl
from gpu_helpers import check_maps, np32, oracle_maps, run_cuda, to_device

pytestmark = pytest.mark.gpu


def _maps(out):
    return [np32(out[k]) for k in ("tok", "frame", "head", "aqf")]


@pytest.mark.parametrize("name", ["tiny", "single", "long65k", "varlen8"])
def test_recompute_maps_match_oracle(cuda_lib, name):
    probe = wl.make_probe(wl.CONFIGS[name])
    out, ws = run_cuda(cuda_lib, probe, text_evidence=True)
    ws.free()
    check_maps(_maps(out), oracle_maps(probe), probe, label=f"{name} recompute")


@pytest.mark.parametrize("name", ["single", "long65k"])
def test_recompute_matches_spill_path(cuda_lib, name):
    probe = wl.make_probe(wl.CONFIGS[name])
    a, ws = run_cuda(cuda_lib, probe)
    ws.free()
    b, ws = run_cuda(cuda_lib, probe, text_evidence=True)
    ws.free()
    for k in ("o", "lse"):
        assert np.array_equal(np32(a[k]), np32(b[k])), k      # the attention itself is unchanged
    for k in ("tok", "frame", "head", "aqf"):
        x, y = np32(a[k]).astype(np.float64), np32(b[k]).astype(np.float64)
        scale = max(np.abs(x).max(), 1e-30)
        assert np.abs(x - y).max() <= 2e-5 * scale, (k, np.abs(x - y).max(), scale)


EDGE = {
    "ragged_tiles_t128_d128": dict(frames=(44,), n_text=(77,), hq=8, hkv=2, d=128, tile=128, window=3),
    "t64_d64_long_text": dict(frames=(36,), n_text=(300,), hq=4, hkv=1, d=64, tile=64, window=2),
    "odd_group_t64": dict(frames=(20,), n_text=(40,), hq=6, hkv=2, d=64, tile=64, window=2),
    "npf64_t128": dict(frames=(9,), n_text=(40,), npf=64, hq=4, hkv=2, d=128, tile=128, window=2),
    "npf4": dict(frames=(70,), n_text=(20,), npf=4, hq=4, hkv=2, d=64, tile=64, window=2),
    "varlen_mixed": dict(frames=(3, 0, 17, 8), n_text=(12, 40, 0, 130), hq=4, hkv=2, d=128, tile=128, window=2),
    "sharp": dict(frames=(40,), n_text=(60,), hq=4, hkv=2, d=128, tile=128, window=4, sharp=True),
}


@pytest.mark.parametrize("name", sorted(EDGE))
def test_recompute_edge_cases(cuda_lib, name):
    from test_gpu_parity import _custom
    probe = _custom(**EDGE[name])
    out, ws = run_cuda(cuda_lib, probe, text_evidence=True)
    ws.free()
    check_maps(_maps(out), oracle_maps(probe), probe, label=f"{name} recompute")


def test_recompute_accumulates_over_layers(cuda_lib):
    cfg = wl.CONFIGS["depth28"]
    mask = wl.build_mask(cfg)
    ws = maps = ref = None
    for layer in range(3):
        probe = wl.make_probe(cfg, layer, mask=mask)
        out, ws = run_cuda(cuda_lib, probe, ws=ws, maps=maps, accumulate=layer > 0, text_evidence=True)
        maps = [out[k] for k in ("tok", "frame", "head", "aqf")]
        r = oracle_maps(probe)
        ref = r if ref is None else [a + b for a, b in zip(ref, r)]
    check_maps([np32(m) for m in maps], ref, probe, label="3 layers recompute")
    ws.free()


def test_noalloc_recompute_fits_the_65k_probe(cuda_lib):
    """Without the spill the 65,664-token probe fits the no-alloc scratch."""
    import torch
    probe = wl.make_probe(wl.CONFIGS["long65k"])
    cfg = probe.cfg
    ref, ws = run_cuda(cuda_lib, probe)
    ws.free()
    q, k, v = to_device(probe)
    n, hq, d = q.shape
    total_vis = int(np.sum(probe.n_vis))
    frames = total_vis // cfg.tokens_per_frame
    o = torch.empty((n, hq, d), dtype=torch.bfloat16, device="cuda")
    lse = torch.empty((hq, n), device="cuda")
    tok = torch.full((hq, total_vis), float("nan"), device="cuda")
    frame = torch.full((hq, frames), float("nan"), device="cuda")
    head = torch.full((1, hq), float("nan"), device="cuda")
    aqf = torch.full((frames,), float("nan"), device="cuda")
    status = B.evisel_probe_evidence_noalloc(q, k, v, probe.cu_seqlens, probe.n_vis, cfg.tokens_per_frame, cfg.tile,
                                             probe.row_ptr, probe.col_idx, o, lse, tok, frame, head, aqf,
                                             text_evidence=True)
    assert status == 0
    assert np.array_equal(o.float().cpu().numpy(), np32(ref["o"]))
    for got, want in ((tok, ref["tok"]), (frame, ref["frame"]), (head, ref["head"]), (aqf, ref["aqf"])):
        x, y = np32(got).astype(np.float64), np32(want).astype(np.float64)
        assert np.all(np.isfinite(x))
        assert np.abs(x - y).max() <= 2e-5 * max(np.abs(y).max(), 1e-30)
