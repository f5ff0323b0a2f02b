"""Float64 oracle: dense masked attention plus explicit probability sums.

TEST INFRASTRUCTURE ONLY (see the package docstring): not part of the product.

The probe computes EXACT masked softmax attention, so this module is the plain
definition written out, one video and one head at a time, in float64 with the
bf16 inputs widened exactly:

  class     token p of a video is visual if p < n_vis, else text
  tile id   visual p -> p // t_s;  text p -> n_vt + (p - n_vis) // t_s,
            n_vt = ceil(n_vis / t_s)      (Appendix, "Detailed Sparse
            Prefilling": frame-aligned visual blocks; query tokens are
            partitioned independently and the last block may be short)
  allowed   (i, j) same video, p_j <= p_i, and i is a text row or
            tile(j) is in the retained set of tile(i)   (Sec. 3.2: block-sparse
            attention restricted to retained blocks; causal history H_i of the
            Appendix is "blocks of the same input sample that precede i")
  logits    s_ij = q_i . k_j / sqrt(d)                   (Eq. 8, token form)
  softmax   LSE_i = ln sum_allowed exp(s_ij) (max-shifted), P_ij = exp(s_ij - LSE_i),
            O_i = sum_j P_ij v_j                           (Eq. 11)
  GQA       query head h reads KV head h // (Hq / Hkv)   (contiguous grouping;
            the paper omits heads, "head indices are omitted for clarity")

Evidence (Sec. 3.2, "Evidence Decomposition"): with P from the text rows,
  tok[h, m]   = sum over text rows i of P_im, for the video's visual tokens m
  frame[h, t] = sum of tok[h, m] over frame t's N_v tokens [t N_v, (t+1) N_v)
  head[b, h]  = sum over the video's frames of frame[h, t]
  A_qf[t]     = sum_h frame[h, t] / (Hq * n_text)   (average over the whole
                query-token group and over heads; 0 for a video without query
                tokens, a case the paper does not have)
With P from the visual rows,
  A_if[t, i, j] = (1 / Hq) sum_h P^h_(t N_v + i, t N_v + j) for j <= i, else 0:
                the token-level causal attention inside frame t, head-averaged
                (the intra-frame cue; P is the row's full softmax over all of
                its allowed keys, so a frame row sums to its in-frame share).
  A_ff[a-1, b]  = (1 / (N_v Hq)) sum_h sum_{i in frame a} sum_{j in frame b} P^h_ij
                for the frames b < a of one video (the cross-frame cue: the
                attention frame a gives to frame b, averaged over a's rows and
                over heads), an array [(T-1), (T-1)] per video, 0 for b >= a
  E_ff[t]       = ( sum_{b<t} A_ff[t-1, b] + sum_{a>t} A_ff[a-1, t] ) / 2: the
                attention frame t gives to earlier frames and the attention it
                receives from later ones, averaged (timestamp-aligned).
"""
from __future__ import annotations

import math

import numpy as np

__all__ = ["token_layout", "allowed_row", "probe_rows", "probe", "text_probabilities", "evidence", "intra_frame"]


def token_layout(n_vis: int, n_text: int, tile: int):
    """(is_text[N], tile_id[N]) for the local positions of one video."""
    n = n_vis + n_text
    p = np.arange(n)
    is_text = p >= n_vis
    n_vt = -(-n_vis // tile)
    tile_id = np.where(is_text, n_vt + (p - n_vis) // tile, p // tile)
    return is_text, tile_id


def _video_csr_rows(cu_seqlens, n_vis, tile, row_ptr, col_idx):
    """Per video, the list of retained kv-tile sets of its visual row tiles."""
    out, r = [], 0
    for b in range(len(n_vis)):
        n_vt = -(-int(n_vis[b]) // tile)
        rows = []
        for _ in range(n_vt):
            rows.append(set(int(c) for c in col_idx[row_ptr[r]:row_ptr[r + 1]]))
            r += 1
        out.append(rows)
    return out


def allowed_row(p: int, is_text, tile_id, retained_rows):
    """Boolean mask over a video's keys for the row at local position p."""
    n = len(is_text)
    j = np.arange(n)
    causal = j <= p
    if is_text[p]:
        return causal
    kept = retained_rows[tile_id[p]]
    assert tile_id[p] in kept, "a visual row tile must retain its diagonal tile"
    keep = np.zeros(int(tile_id.max()) + 1, dtype=bool)
    keep[list(kept)] = True
    return causal & keep[tile_id]


def _attend(qh, kh, vh, allowed, scale):
    """One head, a block of rows: returns (O [r, d], LSE [r], P [r, n]) in float64."""
    s = scale * (qh @ kh.T)
    s = np.where(allowed, s, -np.inf)
    m = s.max(axis=1, keepdims=True)
    assert np.all(np.isfinite(m)), "every row has at least one allowed key"
    e = np.exp(s - m)
    l = e.sum(axis=1, keepdims=True)
    lse = (m + np.log(l))[:, 0]
    p = np.exp(s - lse[:, None])
    o = p @ vh
    return o, lse, p


def probe_rows(q, k, v, cu_seqlens, n_vis, tile, row_ptr, col_idx, rows, scale=None, chunk=512):
    """O and LSE for the global token indices ``rows``.

    Returns (o [len(rows), Hq, d] float64, lse [Hq, len(rows)] float64).
    """
    q = np.asarray(q); k = np.asarray(k); v = np.asarray(v)
    hq, d = q.shape[1], q.shape[2]
    hkv = k.shape[1]
    gq = hq // hkv
    scale = 1.0 / math.sqrt(d) if not scale else float(scale)
    rows = np.asarray(rows, dtype=np.int64)
    cu = np.asarray(cu_seqlens, dtype=np.int64)
    retained = _video_csr_rows(cu, n_vis, tile, row_ptr, col_idx)
    o_out = np.zeros((rows.size, hq, d))
    lse_out = np.zeros((hq, rows.size))
    video_of = np.searchsorted(cu, rows, side="right") - 1
    for b in np.unique(video_of):
        sel = np.nonzero(video_of == b)[0]
        s0, s1 = int(cu[b]), int(cu[b + 1])
        nv = int(n_vis[b])
        is_text, tile_id = token_layout(nv, s1 - s0 - nv, tile)
        kb = k[s0:s1].astype(np.float64)
        vb = v[s0:s1].astype(np.float64)
        for c0 in range(0, sel.size, chunk):
            part = sel[c0:c0 + chunk]
            local = rows[part] - s0
            allowed = np.stack([allowed_row(int(p), is_text, tile_id, retained[b]) for p in local])
            for h in range(hq):
                g = h // gq
                o, lse, _ = _attend(q[rows[part], h, :].astype(np.float64), kb[:, g, :], vb[:, g, :],
                                    allowed, scale)
                o_out[part, h, :] = o
                lse_out[h, part] = lse
    return o_out, lse_out


def probe(q, k, v, cu_seqlens, n_vis, tile, row_ptr, col_idx, scale=None):
    """O [N, Hq, d] and LSE [Hq, N] for every token (small inputs only)."""
    n = np.asarray(q).shape[0]
    return probe_rows(q, k, v, cu_seqlens, n_vis, tile, row_ptr, col_idx, np.arange(n), scale)


def text_probabilities(q, k, cu_seqlens, n_vis, b, h, scale=None):
    """P of video b's text rows for head h: float64 [n_text, N_b] (dense causal rows)."""
    q = np.asarray(q); k = np.asarray(k)
    hq, d = q.shape[1], q.shape[2]
    gq = hq // k.shape[1]
    scale = 1.0 / math.sqrt(d) if not scale else float(scale)
    s0, s1 = int(cu_seqlens[b]), int(cu_seqlens[b + 1])
    nv = int(n_vis[b])
    n = s1 - s0
    pos = np.arange(nv, n)
    allowed = np.arange(n)[None, :] <= pos[:, None]     # text rows see every earlier token
    vdummy = np.zeros((n, 1))
    _, _, p = _attend(q[s0 + nv:s1, h, :].astype(np.float64), k[s0:s1, h // gq, :].astype(np.float64),
                      vdummy, allowed, scale)
    return p


def evidence(q, k, cu_seqlens, n_vis, tokens_per_frame, scale=None):
    """Token, frame, head and query-frame evidence maps from the text rows.

    Returns tok [Hq, sum n_vis], frame [Hq, sum T], head [B, Hq], aqf [sum T]
    (float64). Frames are indexed over the videos in order, T_b = n_vis_b / N_v.
    """
    q = np.asarray(q)
    hq = q.shape[1]
    n_vis = np.asarray(n_vis, dtype=np.int64)
    nb = n_vis.size
    assert np.all(n_vis % tokens_per_frame == 0)
    frames = n_vis // tokens_per_frame
    vis_off = np.concatenate([[0], np.cumsum(n_vis)])
    fr_off = np.concatenate([[0], np.cumsum(frames)])
    tok = np.zeros((hq, int(vis_off[-1])))
    frame = np.zeros((hq, int(fr_off[-1])))
    head = np.zeros((nb, hq))
    aqf = np.zeros(int(fr_off[-1]))
    for b in range(nb):
        nv = int(n_vis[b])
        n_text = int(cu_seqlens[b + 1] - cu_seqlens[b]) - nv
        for h in range(hq):
            p = text_probabilities(q, k, cu_seqlens, n_vis, b, h, scale)
            t_map = p[:, :nv].sum(axis=0)                      # sum over the text rows
            tok[h, vis_off[b]:vis_off[b + 1]] = t_map
            f_map = t_map.reshape(int(frames[b]), tokens_per_frame).sum(axis=1)
            frame[h, fr_off[b]:fr_off[b + 1]] = f_map
            head[b, h] = f_map.sum()
        if n_text > 0:      # a video without query tokens carries no query-frame evidence
            aqf[fr_off[b]:fr_off[b + 1]] = frame[:, fr_off[b]:fr_off[b + 1]].sum(axis=0) / (hq * n_text)
    return tok, frame, head, aqf


def intra_frame(q, k, cu_seqlens, n_vis, tokens_per_frame, tile, row_ptr, col_idx, frames=None, scale=None,
                chunk=512):
    """Intra-frame cue A_if (Sec. 3.2, "Evidence Decomposition"): for frame t
    (global index over the videos in order) the head-averaged causal attention
    among its N_v visual tokens,
        A_if[t, i, j] = (1 / Hq) sum_h P^h_(row i, key j),  j <= i,   0 above,
    where P^h is the probe's probability (the row's softmax over all of its
    allowed keys, Eq. 11). ``frames`` selects global frame indices (default:
    all). Returns float64 [len(frames), N_v, N_v].
    """
    q = np.asarray(q); k = np.asarray(k)
    hq, d = q.shape[1], q.shape[2]
    hkv = k.shape[1]
    gq = hq // hkv
    npf = int(tokens_per_frame)
    scale = 1.0 / math.sqrt(d) if not scale else float(scale)
    n_vis = np.asarray(n_vis, dtype=np.int64)
    cu = np.asarray(cu_seqlens, dtype=np.int64)
    n_frames = n_vis // npf
    fr_off = np.concatenate([[0], np.cumsum(n_frames)])
    frames = np.arange(int(fr_off[-1])) if frames is None else np.asarray(frames, dtype=np.int64)
    retained = _video_csr_rows(cu, n_vis, tile, row_ptr, col_idx)
    out = np.zeros((frames.size, npf, npf))
    video_of = np.searchsorted(fr_off, frames, side="right") - 1
    for b in np.unique(video_of):
        sel = np.nonzero(video_of == b)[0]
        s0, s1 = int(cu[b]), int(cu[b + 1])
        nv = int(n_vis[b])
        is_text, tile_id = token_layout(nv, s1 - s0 - nv, tile)
        kb = k[s0:s1].astype(np.float64)
        # the frames' rows, as local positions
        local = ((frames[sel] - fr_off[b])[:, None] * npf + np.arange(npf)[None, :]).reshape(-1)
        for c0 in range(0, local.size, chunk):
            part = local[c0:c0 + chunk]
            allowed = np.stack([allowed_row(int(p), is_text, tile_id, retained[b]) for p in part])
            for h in range(hq):
                _, _, p = _attend(q[s0 + part, h, :].astype(np.float64), kb[:, h // gq, :],
                                  np.zeros((s1 - s0, 1)), allowed, scale)
                for r, pos in enumerate(part):
                    f = int(pos) // npf          # frame (video-local) of this row
                    i = int(pos) % npf
                    slot = sel[int(np.nonzero((frames[sel] - fr_off[b]) == f)[0][0])]
                    out[slot, i, :] += p[r, f * npf:(f + 1) * npf] / hq
    return out


def frame_mass_rows(q, k, cu_seqlens, n_vis, tokens_per_frame, tile, row_ptr, col_idx, frames, scale=None,
                    chunk=512):
    """For each global frame index a in ``frames``: the attention its visual
    rows give to every frame b of the same video, averaged over the frame's
    N_v rows and over heads,
        M[a, b] = (1 / (N_v Hq)) sum_h sum_{i in a} sum_{j in b} P^h_ij,
    with P the probe's probability (Eq. 11; the row's softmax over all of its
    allowed keys). Returns a list of float64 vectors, one of length T_video
    per requested frame (entries b > a are 0 by causality; b = a is the
    in-frame share)."""
    q = np.asarray(q); k = np.asarray(k)
    hq, d = q.shape[1], q.shape[2]
    hkv = k.shape[1]
    gq = hq // hkv
    npf = int(tokens_per_frame)
    scale = 1.0 / math.sqrt(d) if not scale else float(scale)
    n_vis = np.asarray(n_vis, dtype=np.int64)
    cu = np.asarray(cu_seqlens, dtype=np.int64)
    n_frames = n_vis // npf
    fr_off = np.concatenate([[0], np.cumsum(n_frames)])
    frames = np.asarray(frames, dtype=np.int64)
    retained = _video_csr_rows(cu, n_vis, tile, row_ptr, col_idx)
    video_of = np.searchsorted(fr_off, frames, side="right") - 1
    out = [np.zeros(int(n_frames[b])) for b in video_of]
    for b in np.unique(video_of):
        sel = np.nonzero(video_of == b)[0]
        s0, s1 = int(cu[b]), int(cu[b + 1])
        nv = int(n_vis[b])
        tb = int(n_frames[b])
        is_text, tile_id = token_layout(nv, s1 - s0 - nv, tile)
        kb = k[s0:s1].astype(np.float64)
        local = ((frames[sel] - fr_off[b])[:, None] * npf + np.arange(npf)[None, :]).reshape(-1)
        slot_of_frame = {int(frames[i] - fr_off[b]): int(i) for i in sel}
        for c0 in range(0, local.size, chunk):
            part = local[c0:c0 + chunk]
            allowed = np.stack([allowed_row(int(p), is_text, tile_id, retained[b]) for p in part])
            for h in range(hq):
                _, _, p = _attend(q[s0 + part, h, :].astype(np.float64), kb[:, h // gq, :],
                                  np.zeros((s1 - s0, 1)), allowed, scale)
                # mass of each row on each frame b' of the video (visual keys only)
                per_frame = p[:, :tb * npf].reshape(len(part), tb, npf).sum(axis=2)
                for r, pos in enumerate(part):
                    out[slot_of_frame[int(pos) // npf]] += per_frame[r] / (npf * hq)
    return out


def cross_frame(q, k, cu_seqlens, n_vis, tokens_per_frame, tile, row_ptr, col_idx, scale=None, chunk=512):
    """Cross-frame cue A_ff and its timestamp-aligned evidence E_ff (Sec. 3.2,
    "Evidence Decomposition").

    Returns (aff, eff): ``aff`` a list over videos of float64 [(T-1), (T-1)]
    arrays with aff[a-1, b] = M[a, b] for b < a (M from ``frame_mass_rows``)
    and 0 elsewhere; ``eff`` float64 [sum T] in video order, from ``e_ff``."""
    n_vis = np.asarray(n_vis, dtype=np.int64)
    npf = int(tokens_per_frame)
    n_frames = n_vis // npf
    fr_off = np.concatenate([[0], np.cumsum(n_frames)])
    aff = []
    for b in range(len(n_vis)):
        tb = int(n_frames[b])
        a_b = np.zeros((max(tb - 1, 0), max(tb - 1, 0)))
        if tb > 1:
            rows = frame_mass_rows(q, k, cu_seqlens, n_vis, npf, tile, row_ptr, col_idx,
                                   np.arange(fr_off[b] + 1, fr_off[b] + tb), scale=scale, chunk=chunk)
            for a in range(1, tb):
                a_b[a - 1, :a] = rows[a - 1][:a]
        aff.append(a_b)
    return aff, e_ff(aff, n_frames)


def e_ff(aff, n_frames):
    """E_ff from A_ff: for frame t of a video with T frames,
        E_ff[t] = ( sum_{b<t} A_ff[t-1, b] + sum_{a>t} A_ff[a-1, t] ) / 2
    (the attention t gives to earlier frames, row t-1 of A_ff, and the
    attention it receives from later frames, column t); an empty side is an
    empty sum. Returns float64 [sum T]."""
    out = []
    for a_b, tb in zip(aff, n_frames):
        tb = int(tb)
        e = np.zeros(tb)
        for t in range(tb):
            give = a_b[t - 1, :t].sum() if t >= 1 else 0.0
            recv = a_b[t:, t].sum() if t <= tb - 2 else 0.0     # rows a-1 = t .. T-2, i.e. frames a = t+1 .. T-1
            e[t] = 0.5 * (give + recv)
        out.append(e)
    return np.concatenate(out) if out else np.zeros(0)
