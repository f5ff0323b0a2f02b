"""Seeded synthetic inputs for the sparse-prefill evidence probe.

This module is the only code shared by the CUDA path's tests/bench and the
float64 oracle. It draws inputs and builds the block mask; it holds none of the
probe's arithmetic (no logits, no softmax, no evidence sums).

Shapes follow the probe's context layout X = [X_vis; X_Q] (paper Sec. 3.2 and
Appendix "Detailed Sparse Prefilling"): per video, n_vis = T * N_v pooled
visual tokens followed by n_text query tokens, packed back to back over
videos (varlen, ``cu_seqlens``). Q is [N_tot, Hq, d], K and V are
[N_tot, Hkv, d], all bf16-representable values (kept here as float32).

Tile partition (Appendix, frame-aligned blocks): visual tokens of a video are
cut into tiles of ``tile`` tokens from the visual start (the last may be
short); text tokens are cut independently from the text start. ``tile`` is a
multiple of N_v, so no frame crosses a tile. The mask is a CSR over the
visual row tiles of all videos (video order), each row a sorted list of
video-local visual kv-tile ids; text rows are implicitly dense-causal.

Mask recipe (static stand-in for top-p retention): each visual row tile r
keeps the sink tile 0, the causal window {r-W+1..r} clipped at 0, and
optionally ``extra`` random causal tiles drawn from {1..r-1} minus the
already kept ones (without replacement, one generator consumed row by row).

Planting: a planted frame's keys get 2 * u_g added, u_g being the float32
mean of Q over the video's text rows and the query heads of KV group g
(contiguous grouping, g = h // (Hq / Hkv)), before bf16 rounding.
"""
from __future__ import annotations

from dataclasses import dataclass, field
import math

import numpy as np

__all__ = [
    "ProbeConfig", "CONFIGS", "Probe", "make_probe", "bf16_round",
    "build_mask", "video_tiles", "config_by_name",
]


def bf16_round(x: np.ndarray, inplace: bool = False) -> np.ndarray:
    """Round float32 values to the nearest bfloat16 (ties to even); returns float32."""
    if not (inplace and x.dtype == np.float32 and x.flags.c_contiguous):
        x = np.array(x, dtype=np.float32, copy=True, order="C")
    flat = x.reshape(-1).view(np.uint32)
    step = 1 << 18                              # cache-sized chunks, finite inputs (no uint32 overflow)
    lsb = np.empty(step, np.uint32)
    for a in range(0, flat.size, step):
        u = flat[a:a + step]
        r = lsb[:u.size]
        np.right_shift(u, 16, out=r)
        np.bitwise_and(r, 1, out=r)
        r += np.uint32(0x7FFF)
        u += r
        u &= np.uint32(0xFFFF0000)
    return x


@dataclass(frozen=True)
class ProbeConfig:
    """One synthetic probe workload (one or more independent layers)."""
    name: str
    frames: tuple          # frames T_b per video
    tokens_per_frame: int  # N_v
    n_text: tuple          # query tokens per video
    hq: int
    hkv: int
    head_dim: int
    tile: int
    window: int            # causal window W in tiles (includes the diagonal)
    extra: int = 0         # random extra causal tiles per visual row tile
    plant: tuple = ()      # planted frames per video (count)
    layers: int = 1
    seed: int = 0
    mask_seed: int | None = None
    qkv_seed: object = None   # seed for Q/K/V draws (default: ``seed``)
    scale_inputs: bool = True  # Q/K/V ~ N(0,1)/sqrt(d); False gives "sharp" N(0,1)
    description: str = ""
    # "clustered": concentrated attention (see _clustered); default: i.i.d. draws
    regime: str = "iid"

    @property
    def n_vis(self):
        return tuple(f * self.tokens_per_frame for f in self.frames)

    @property
    def seqlens(self):
        return tuple(a + b for a, b in zip(self.n_vis, self.n_text))

    @property
    def n_tot(self):
        return sum(self.seqlens)

    @property
    def num_videos(self):
        return len(self.frames)


def _plant_count(frac, frames):
    return tuple(max(1, int(round(frac * t))) for t in frames)


def _c5_lengths():
    rng = np.random.default_rng(4)
    frames = rng.integers(512, 2049, 8)
    text = rng.integers(64, 257, 8)
    return tuple(int(x) for x in frames), tuple(int(x) for x in text)


_C5_FRAMES, _C5_TEXT = _c5_lengths()

CONFIGS = {
    "tiny": ProbeConfig(
        "tiny", (32,), 16, (32,), 4, 2, 64, 64, 2, plant=(3,), seed=0,
        description="32 frames x 16 tokens + 32 text; 4q/2kv, d=64; 64-tiles, sink+2-window"),
    "single": ProbeConfig(
        "single", (256,), 16, (64,), 28, 4, 128, 128, 4, plant=_plant_count(0.05, (256,)), seed=1,
        description="256 frames x 16 tokens + 64 text; 28q/4kv, d=128; 128-tiles, sink+4-window"),
    "depth28": ProbeConfig(
        "depth28", (1024,), 16, (128,), 28, 4, 128, 128, 8, plant=_plant_count(0.05, (1024,)),
        layers=28, seed=2,
        description="28 layers of 1024 frames x 16 tokens + 128 text; 28q/4kv, d=128; sink+8-window"),
    "long65k": ProbeConfig(
        "long65k", (1024,), 64, (128,), 28, 4, 128, 128, 16, extra=32,
        plant=_plant_count(0.02, (1024,)), seed=3, mask_seed=3,
        description="1024 frames x 64 tokens + 128 text (65,664 tokens); 28q/4kv, d=128; "
                    "sink+16-window+32 random tiles per visual row tile"),
    "prof24k": ProbeConfig(
        "prof24k", (384,), 64, (128,), 28, 4, 128, 128, 16, extra=32,
        plant=_plant_count(0.02, (384,)), seed=3, mask_seed=3,
        description="profiling-size variant of long65k: 384 frames x 64 tokens + 128 text (24,704 tokens); "
                    "same heads, tiles and mask recipe; inputs still larger than L2"),
    "long65k_sparse": ProbeConfig(
        "long65k_sparse", (1024,), 64, (128,), 28, 4, 128, 128, 16, extra=32, seed=5, mask_seed=3,
        scale_inputs=False, regime="clustered",
        description="long65k's shapes with concentrated attention (clustered keys and queries, see "
                    "_clustered): the regime where top-p retention keeps a small share of each row's history"),
    "varlen8": ProbeConfig(
        "varlen8", _C5_FRAMES, 16, _C5_TEXT, 28, 4, 128, 128, 8,
        plant=_plant_count(0.05, _C5_FRAMES), seed=4, qkv_seed=(4, 1),
        description="8 packed videos, 512-2048 frames x 16 tokens + 64-256 text; 28q/4kv, d=128; sink+8-window"),
}


def config_by_name(name: str) -> ProbeConfig:
    return CONFIGS[name]


def video_tiles(n_vis: int, n_text: int, tile: int):
    """Return (number of visual tiles, number of text tiles) of one video."""
    return -(-n_vis // tile), -(-n_text // tile)


def build_mask(cfg: ProbeConfig):
    """CSR (row_ptr, col_idx) over the visual row tiles of all videos."""
    rng = np.random.default_rng(cfg.mask_seed) if cfg.extra else None
    row_ptr = [0]
    cols = []
    for n_vis, n_text in zip(cfg.n_vis, cfg.n_text):
        n_vt, _ = video_tiles(n_vis, n_text, cfg.tile)
        for r in range(n_vt):
            kept = {0} | set(range(max(0, r - cfg.window + 1), r + 1))
            if cfg.extra:
                cand = np.array([c for c in range(1, r) if c not in kept], dtype=np.int64)
                take = min(cfg.extra, cand.size)
                if take:
                    kept |= set(int(c) for c in rng.choice(cand, size=take, replace=False))
            cols.extend(sorted(kept))
            row_ptr.append(len(cols))
    return np.asarray(row_ptr, dtype=np.int32), np.asarray(cols, dtype=np.int32)


@dataclass
class Probe:
    """Materialised inputs of one layer of a config."""
    cfg: ProbeConfig
    layer: int
    q: np.ndarray            # float32 [N_tot, Hq, d], bf16-representable
    k: np.ndarray            # float32 [N_tot, Hkv, d]
    v: np.ndarray            # float32 [N_tot, Hkv, d]
    cu_seqlens: np.ndarray   # int32 [B+1]
    n_vis: np.ndarray        # int32 [B]
    row_ptr: np.ndarray      # int32 CSR over visual row tiles
    col_idx: np.ndarray      # int32 video-local kv tile ids
    planted: list = field(default_factory=list)   # per video: sorted planted frame ids

    @property
    def n_text(self):
        return np.diff(self.cu_seqlens) - self.n_vis


def _planted_frames(cfg: ProbeConfig):
    rng = np.random.default_rng([cfg.seed, 99])
    out = []
    for t, cnt in zip(cfg.frames, cfg.plant or (0,) * cfg.num_videos):
        out.append(np.sort(rng.choice(t, size=cnt, replace=False)).astype(np.int64) if cnt else
                   np.zeros(0, np.int64))
    return out


CLUSTER_KEY_WEIGHT = 3.0      # alpha: weight of a block's topic in its keys
CLUSTER_QUERY_NOISE = 0.25    # gamma: weight of a query's own noise
CLUSTER_RECENT = 4            # targets of a row tile: its most recent earlier blocks ...
CLUSTER_RANDOM = 4            # ... and this many random earlier blocks


def _clustered(cfg: ProbeConfig, q, k, cu, rng):
    """Concentrated attention (a stand-in for the regime where top-p retention
    keeps few blocks): every block of N_v tokens of a video has a topic vector
    c_j ~ N(0, I_d) per KV group, and its keys are alpha c_j + N(0, I_d); every
    query row tile (tiles of ``cfg.tile`` rows over the visual rows, then over
    the text rows) draws target blocks among the blocks that end before it (its
    CLUSTER_RECENT most recent ones and CLUSTER_RANDOM random earlier ones),
    and its queries are s + gamma N(0, I_d) with s the targets' topics summed
    and divided by sqrt(#targets) (per KV group, shared by the group's heads).
    ``q`` and ``k`` hold the N(0, 1) draws on entry and are overwritten."""
    d, npf, T = cfg.head_dim, cfg.tokens_per_frame, cfg.tile
    gq = cfg.hq // cfg.hkv
    for b in range(cfg.num_videos):
        s0, nv, nt = int(cu[b]), cfg.n_vis[b], cfg.n_text[b]
        n_blk = nv // npf + -(-nt // npf)
        topic = rng.standard_normal((n_blk, cfg.hkv, d), dtype=np.float32)
        blk_of = np.concatenate([np.arange(nv) // npf, nv // npf + np.arange(nt) // npf])
        k[s0:s0 + nv + nt] = np.float32(CLUSTER_KEY_WEIGHT) * topic[blk_of] + k[s0:s0 + nv + nt]
        starts = [(t * T, min(T, nv - t * T)) for t in range(-(-nv // T))]
        starts += [(nv + t * T, min(T, nt - t * T)) for t in range(-(-nt // T))]
        ends = np.array([min(j * npf + npf, nv) if j < nv // npf else nv + (j - nv // npf + 1) * npf
                         for j in range(n_blk)])
        for a, n in starts:
            hist = np.nonzero(ends <= a)[0]               # blocks that end before the tile's first row
            if hist.size == 0:
                tgt = np.zeros(0, np.int64)
            else:
                recent = hist[-CLUSTER_RECENT:]
                rest = hist[:-CLUSTER_RECENT] if hist.size > CLUSTER_RECENT else hist[:0]
                pick = rng.choice(rest, size=min(CLUSTER_RANDOM, rest.size), replace=False) if rest.size else rest
                tgt = np.concatenate([recent, pick])
            rows = slice(s0 + a, s0 + a + n)
            noise = np.float32(CLUSTER_QUERY_NOISE) * q[rows]
            if tgt.size:
                centre = topic[tgt].sum(axis=0) / np.float32(math.sqrt(tgt.size))   # [hkv, d]
                q[rows] = noise + np.repeat(centre, gq, axis=0)[None]
            else:
                q[rows] = noise


def make_probe(cfg: ProbeConfig, layer: int = 0, mask=None) -> Probe:
    """Draw Q/K/V for one layer of ``cfg`` and return them with the mask."""
    if cfg.layers > 1:
        seed = [cfg.seed, layer]
    elif cfg.qkv_seed is not None:
        seed = list(cfg.qkv_seed) if isinstance(cfg.qkv_seed, tuple) else cfg.qkv_seed
    else:
        seed = cfg.seed
    rng = np.random.default_rng(seed)
    n, d = cfg.n_tot, cfg.head_dim
    div = np.float32(math.sqrt(d)) if cfg.scale_inputs else np.float32(1.0)
    q = rng.standard_normal((n, cfg.hq, d), dtype=np.float32)
    k = rng.standard_normal((n, cfg.hkv, d), dtype=np.float32)
    v = rng.standard_normal((n, cfg.hkv, d), dtype=np.float32)
    for x in (q, k, v):
        np.divide(x, div, out=x)
    cu = np.zeros(cfg.num_videos + 1, dtype=np.int64)
    cu[1:] = np.cumsum(cfg.seqlens)
    if cfg.regime == "clustered":
        _clustered(cfg, q, k, cu, np.random.default_rng([cfg.seed, 7]))
    planted = _planted_frames(cfg)
    gq = cfg.hq // cfg.hkv
    nv_tok = cfg.tokens_per_frame
    for b in range(cfg.num_videos):
        if planted[b].size == 0:
            continue
        s, nv = int(cu[b]), cfg.n_vis[b]
        text_q = q[s + nv:int(cu[b + 1])]                     # [n_text, Hq, d]
        for g in range(cfg.hkv):
            u = text_q[:, g * gq:(g + 1) * gq, :].reshape(-1, d).mean(axis=0, dtype=np.float32)
            for f in planted[b]:
                a = s + int(f) * nv_tok
                k[a:a + nv_tok, g, :] += np.float32(2.0) * u
    if mask is None:
        mask = build_mask(cfg)
    row_ptr, col_idx = mask
    return Probe(cfg, layer, bf16_round(q, True), bf16_round(k, True), bf16_round(v, True),
                 cu.astype(np.int32), np.asarray(cfg.n_vis, dtype=np.int32),
                 row_ptr, col_idx, planted)
