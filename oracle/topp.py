"""Float64 oracle of the paper's top-p block retention (Appendix, "Detailed
Sparse Prefilling", Eq. 6-9 and the retention rule after Eq. 9).

TEST INFRASTRUCTURE ONLY (see the package docstring): not part of the product.

  blocks    per video: visual blocks of B tokens from the visual start (B
            divides N_v, so no block crosses a frame), then the text tokens
            cut into blocks of B from the text start (the last may be short);
            block ids count the visual blocks first
  k_bar_j   mean of the block's keys, per KV head                    (Eq. 7)
  H_i       the blocks of the row's video that end before position i
            (last token < i); the row's own block is never in H_i
  g_ij      q_i . k_bar_j / sqrt(d) for j in H_i                      (Eq. 8)
  p_ij      softmax of g_i. over H_i                                  (Eq. 9)
  S_i       H_i ordered by p descending (ties: lower block id first), the
            shortest prefix whose cumulative p reaches tau_p
  attended  the tokens of the blocks in S_i, and the causal prefix of the
            row's own block (the row's E_i; there is no system prefix here)
Head h reads KV head h // (Hq / Hkv).
"""
from __future__ import annotations

import math

import numpy as np


def block_layout(n_vis: int, n_text: int, block: int):
    """(start, length) of every block of one video, in block-id order."""
    out = [(s, block) for s in range(0, n_vis, block)]
    out += [(n_vis + s, min(block, n_text - s)) for s in range(0, n_text, block)]
    return out


def block_means(k_video, n_vis: int, n_text: int, block: int):
    """k_bar [n_blocks, Hkv, d] float64 for one video: the mean of each
    block's keys (Eq. 7)."""
    k = np.asarray(k_video, dtype=np.float64)
    return np.stack([k[s:s + n].mean(axis=0) for s, n in block_layout(n_vis, n_text, block)])


def select_prefix(p, tau):
    """Indices (into p) of the shortest prefix of p ordered descending (ties:
    lower index first) whose cumulative sum reaches tau."""
    order = sorted(range(len(p)), key=lambda j: (-p[j], j))
    acc, keep = 0.0, []
    for j in order:
        if acc >= tau:
            break
        keep.append(j)
        acc += p[j]
    return sorted(keep)


def retained_blocks(q, k, cu_seqlens, n_vis, block, tau_p, rows=None, heads=None, scale=None):
    """S_i for the global token indices ``rows`` (default: all) and query heads
    ``heads`` (default: all). Returns a dict {(h, row): sorted list of the
    video's block ids}, and the matching p_i. as {(h, row): (block ids of H_i,
    p over them)}."""
    q = np.asarray(q); k = np.asarray(k)
    n, hq, d = q.shape
    gq = hq // k.shape[1]
    scale = 1.0 / math.sqrt(d) if not scale else float(scale)
    cu = np.asarray(cu_seqlens, dtype=np.int64)
    n_vis = np.asarray(n_vis, dtype=np.int64)
    rows = np.arange(int(cu[-1])) if rows is None else np.asarray(rows, dtype=np.int64)
    heads = range(hq) if heads is None else heads
    sets, probs = {}, {}
    video_of = np.searchsorted(cu, rows, side="right") - 1
    for b in np.unique(video_of):
        s0, s1, nv = int(cu[b]), int(cu[b + 1]), int(n_vis[b])
        layout = block_layout(nv, s1 - s0 - nv, block)
        kbar = block_means(k[s0:s1], nv, s1 - s0 - nv, block)
        ends = np.array([s + ln for s, ln in layout])           # one past each block's last token
        for row in rows[video_of == b]:
            p_loc = int(row) - s0
            hist = np.nonzero(ends <= p_loc)[0]                  # blocks that end before the row
            for h in heads:
                if hist.size == 0:
                    sets[(h, int(row))] = []
                    probs[(h, int(row))] = (hist, np.zeros(0))
                    continue
                g = scale * (kbar[hist, h // gq, :] @ q[row, h, :].astype(np.float64))
                e = np.exp(g - g.max())
                p = e / e.sum()
                keep = select_prefix(list(p), tau_p)
                sets[(h, int(row))] = [int(hist[j]) for j in keep]
                probs[(h, int(row))] = (hist, p)
    return sets, probs


def attended_mask(row_local: int, n_vis: int, n_text: int, block: int, kept):
    """Boolean mask over the video's keys for a row at local position
    ``row_local`` with retained blocks ``kept``: the kept blocks' tokens and
    the causal prefix of the row's own block."""
    layout = block_layout(n_vis, n_text, block)
    n = n_vis + n_text
    mask = np.zeros(n, dtype=bool)
    for j in kept:
        s, ln = layout[j]
        mask[s:s + ln] = True
    own = next(j for j, (s, ln) in enumerate(layout) if s <= row_local < s + ln)
    s, _ = layout[own]
    mask[s:row_local + 1] = True
    return mask


def probe_rows_topp(q, k, v, cu_seqlens, n_vis, block, kept, rows, scale=None):
    """O [len(rows), Hq, d] and LSE [Hq, len(rows)] (float64) of the rows
    attending to their retained blocks ``kept`` ({(h, row): block ids}) and
    their own block's causal prefix (the sparse prefill of Eq. 1 with the
    top-p masks)."""
    q = np.asarray(q); k = np.asarray(k); v = np.asarray(v)
    n, hq, d = q.shape
    gq = hq // k.shape[1]
    scale = 1.0 / math.sqrt(d) if not scale else float(scale)
    cu = np.asarray(cu_seqlens, dtype=np.int64)
    n_vis = np.asarray(n_vis, dtype=np.int64)
    rows = np.asarray(rows, dtype=np.int64)
    o = np.zeros((rows.size, hq, v.shape[2]))
    lse = np.zeros((hq, rows.size))
    for r, row in enumerate(rows):
        b = int(np.searchsorted(cu, row, side="right") - 1)
        s0, s1, nv = int(cu[b]), int(cu[b + 1]), int(n_vis[b])
        for h in range(hq):
            m = attended_mask(int(row) - s0, nv, s1 - s0 - nv, block, kept[(h, int(row))])
            s = scale * (k[s0:s1, h // gq, :].astype(np.float64) @ q[row, h, :].astype(np.float64))
            s = np.where(m, s, -np.inf)
            mx = s.max()
            w = np.exp(s - mx)
            lse[h, r] = mx + math.log(w.sum())
            o[r, h, :] = (w / w.sum()) @ v[s0:s1, h // gq, :].astype(np.float64)
    return o, lse


def evidence_topp(q, k, cu_seqlens, n_vis, tokens_per_frame, block, kept, scale=None):
    """The evidence maps of the text rows attending to their retained blocks
    ``kept`` ({(h, row): block ids}) and their own block's causal prefix:
    P_im = exp(s_im - LSE_i) over the attended keys, summed over the text rows
    into tok [Hq, sum n_vis], then frame [Hq, sum T], head [B, Hq] and
    aqf [sum T] as in the dense evidence (Sec. 3.2)."""
    q = np.asarray(q); k = np.asarray(k)
    n, hq, d = q.shape
    gq = hq // k.shape[1]
    scale = 1.0 / math.sqrt(d) if not scale else float(scale)
    cu = np.asarray(cu_seqlens, dtype=np.int64)
    n_vis = np.asarray(n_vis, dtype=np.int64)
    npf = int(tokens_per_frame)
    frames = n_vis // npf
    vis_off = np.concatenate([[0], np.cumsum(n_vis)])
    fr_off = np.concatenate([[0], np.cumsum(frames)])
    tok = np.zeros((hq, int(vis_off[-1])))
    frame = np.zeros((hq, int(fr_off[-1])))
    head = np.zeros((len(n_vis), hq))
    aqf = np.zeros(int(fr_off[-1]))
    for b in range(len(n_vis)):
        s0, s1, nv = int(cu[b]), int(cu[b + 1]), int(n_vis[b])
        n_text = s1 - s0 - nv
        for h in range(hq):
            t_map = np.zeros(nv)
            for row in range(s0 + nv, s1):
                m = attended_mask(row - s0, nv, n_text, block, kept[(h, row)])
                s = scale * (k[s0:s1, h // gq, :].astype(np.float64) @ q[row, h, :].astype(np.float64))
                s = np.where(m, s, -np.inf)
                mx = s.max()
                p = np.exp(s - mx)
                p /= p.sum()
                t_map += p[:nv]
            tok[h, vis_off[b]:vis_off[b + 1]] = t_map
            f_map = t_map.reshape(int(frames[b]), npf).sum(axis=1)
            frame[h, fr_off[b]:fr_off[b + 1]] = f_map
            head[b, h] = f_map.sum()
        if n_text > 0:
            aqf[fr_off[b]:fr_off[b + 1]] = frame[:, fr_off[b]:fr_off[b + 1]].sum(axis=0) / (hq * n_text)
    return tok, frame, head, aqf


def coarse_evidence(q, k, cu_seqlens, n_vis, tokens_per_frame, block, kept, scale=None):
    """Evidence maps from the coarse token-level map (Appendix Eq. 10-11): for a
    text row i, a_im = q_i k_m / sqrt(d) for the keys m of its own block up to
    i (E_i; there is no system prefix here), a_im = g_ij for the tokens of each
    retained block K_j in S_i = ``kept[(h, row)]``, -inf elsewhere; the map is
    the row softmax of a. Its mass on the visual tokens is summed over the
    text rows into tok [Hq, sum n_vis], then frame, head and aqf as in the
    exact evidence (Sec. 3.2)."""
    q = np.asarray(q); k = np.asarray(k)
    n, hq, d = q.shape
    gq = hq // k.shape[1]
    scale = 1.0 / math.sqrt(d) if not scale else float(scale)
    cu = np.asarray(cu_seqlens, dtype=np.int64)
    n_vis = np.asarray(n_vis, dtype=np.int64)
    npf = int(tokens_per_frame)
    frames = n_vis // npf
    vis_off = np.concatenate([[0], np.cumsum(n_vis)])
    fr_off = np.concatenate([[0], np.cumsum(frames)])
    tok = np.zeros((hq, int(vis_off[-1])))
    frame = np.zeros((hq, int(fr_off[-1])))
    head = np.zeros((len(n_vis), hq))
    aqf = np.zeros(int(fr_off[-1]))
    for b in range(len(n_vis)):
        s0, s1, nv = int(cu[b]), int(cu[b + 1]), int(n_vis[b])
        n_text = s1 - s0 - nv
        layout = block_layout(nv, n_text, block)
        kbar = block_means(k[s0:s1], nv, n_text, block)
        for h in range(hq):
            t_map = np.zeros(nv)
            for row in range(s0 + nv, s1):
                pos = row - s0
                qv = q[row, h, :].astype(np.float64)
                a = np.full(s1 - s0, -np.inf)
                for j in kept[(h, row)]:
                    s, ln = layout[j]
                    a[s:s + ln] = scale * float(kbar[j, h // gq, :] @ qv)
                own = next(j for j, (s, ln) in enumerate(layout) if s <= pos < s + ln)
                so, _ = layout[own]
                a[so:pos + 1] = scale * (k[s0 + so:s0 + pos + 1, h // gq, :].astype(np.float64) @ qv)
                w = np.exp(a - a.max())
                t_map += (w / w.sum())[:nv]
            tok[h, vis_off[b]:vis_off[b + 1]] = t_map
            f_map = t_map.reshape(int(frames[b]), npf).sum(axis=1)
            frame[h, fr_off[b]:fr_off[b + 1]] = f_map
            head[b, h] = f_map.sum()
        if n_text > 0:
            aqf[fr_off[b]:fr_off[b + 1]] = frame[:, fr_off[b]:fr_off[b + 1]].sum(axis=0) / (hq * n_text)
    return tok, frame, head, aqf
