"""Shared helpers of the GPU parity tests: run the CUDA path through the C ABI
binding and compare it with the float64 oracle at the stated tolerances.

Tolerances (float64 oracle vs the bf16-in / bf16-out kernel):
  O      max abs <= 2e-2 and relative L2 <= 5e-3
  LSE    max abs <= 1e-3
  maps   frame map: max abs <= 1e-3 per entry, on the raw sums (over text
         rows, and over layers where the maps accumulate), as the contract
         states it for frame evidence; the token map at the same bound;
         A_qf (an average over text rows and heads, summed over layers):
         max abs <= 1e-3;
         head map: relative error <= 1e-3 (each entry is a sum of
         probabilities exp(s - LSE), so an LSE within 1e-3 moves it by at
         most a factor e^(1e-3)); identical planted top-k on the head-summed
         frame map.
"""
import numpy as np

import oracle

O_MAX_ABS = 2e-2
O_REL_L2 = 5e-3
LSE_ABS = 1e-3
MAP_ABS = 1e-3
HEAD_REL = 1e-3


def to_device(probe):
    import torch
    dev = dict(device="cuda")
    q = torch.from_numpy(probe.q).to(**dev).to(torch.bfloat16).contiguous()
    k = torch.from_numpy(probe.k).to(**dev).to(torch.bfloat16).contiguous()
    v = torch.from_numpy(probe.v).to(**dev).to(torch.bfloat16).contiguous()
    return q, k, v


def run_cuda(ev, probe, ws=None, maps=None, accumulate=False, qkv=None, text_evidence=False):
    """Probe + evidence on the GPU; returns numpy outputs and the workspace.
    ``text_evidence``: the evidence recomputed from q and k instead of the spill."""
    import torch
    cfg = probe.cfg
    q, k, v = qkv if qkv is not None else to_device(probe)
    o, lse, ws = ev.evisel_probe_attention(q, k, v, probe.cu_seqlens, probe.n_vis, cfg.tokens_per_frame,
                                           cfg.tile, probe.row_ptr, probe.col_idx, ws=ws,
                                           text_evidence=text_evidence)
    kw = {}
    if maps is not None:
        kw = dict(tok=maps[0], frame=maps[1], head=maps[2], aqf=maps[3])
    tok, frame, head, aqf = ev.evisel_evidence_reduce(ws, cfg.hq, probe.n_vis, cfg.tokens_per_frame,
                                                      len(probe.n_vis), accumulate=accumulate, **kw)
    torch.cuda.synchronize()
    assert ev.evisel_status(ws) == 0
    return dict(o=o, lse=lse, tok=tok, frame=frame, head=head, aqf=aqf), ws


def np32(t):
    return t.float().cpu().numpy()


def check_o(o_gpu, o_ref, label=""):
    o_gpu = np.asarray(o_gpu, dtype=np.float64)
    err = np.abs(o_gpu - o_ref)
    rel = np.linalg.norm(o_gpu - o_ref) / max(np.linalg.norm(o_ref), 1e-30)
    assert np.all(np.isfinite(o_gpu)), f"{label}: non-finite O"
    assert err.max() <= O_MAX_ABS, f"{label}: O max abs {err.max():.3e}"
    assert rel <= O_REL_L2, f"{label}: O rel L2 {rel:.3e}"
    return err.max(), rel


def check_lse(lse_gpu, lse_ref, label=""):
    err = np.abs(np.asarray(lse_gpu, np.float64) - lse_ref)
    assert np.all(np.isfinite(lse_gpu)), f"{label}: non-finite LSE"
    assert err.max() <= LSE_ABS, f"{label}: LSE max abs {err.max():.3e}"
    return err.max()


def oracle_maps(probe):
    return oracle.evidence(probe.q, probe.k, probe.cu_seqlens, probe.n_vis, probe.cfg.tokens_per_frame)


def check_maps(gpu, ref, probe, label=""):
    """Compares the raw maps (sums over layers on both sides where they accumulate)."""
    tok, frame, head, aqf = (np.asarray(x, np.float64) for x in gpu)
    rtok, rframe, rhead, raqf = (np.asarray(x, np.float64) for x in ref)
    cfg = probe.cfg
    frames = probe.n_vis // cfg.tokens_per_frame
    e_tok = np.abs(tok - rtok)
    e_fr = np.abs(frame - rframe)
    e_head = np.abs(head - rhead) / np.maximum(np.abs(rhead), 1e-30)
    e_head = np.where(np.abs(rhead) > 0, e_head, np.abs(head - rhead))
    e_aqf = np.abs(aqf - raqf)
    for name, e, bound in (("tok", e_tok, MAP_ABS), ("frame", e_fr, MAP_ABS), ("head (relative)", e_head, HEAD_REL),
                           ("aqf", e_aqf, MAP_ABS)):
        if e.size:
            assert np.all(np.isfinite(e)), f"{label}: non-finite {name}"
            assert e.max() <= bound, f"{label}: {name} max error {e.max():.3e}"
    # planted frames: identical top-k on the head-summed frame map, per video
    off = 0
    for b, planted in enumerate(probe.planted):
        nf = int(frames[b])
        if planted.size:
            g = frame[:, off:off + nf].sum(axis=0)
            r = rframe[:, off:off + nf].sum(axis=0)
            kk = planted.size
            top_g = np.sort(np.argsort(-g, kind="stable")[:kk])
            top_r = np.sort(np.argsort(-r, kind="stable")[:kk])
            np.testing.assert_array_equal(top_g, top_r, err_msg=f"{label}: top-k frames of video {b}")
        off += nf
    return max(e.max() if e.size else 0 for e in (e_tok, e_fr, e_aqf))
