"""Benchmark of the sparse-prefill evidence probe on one GB300 (or N replicas).

One step = the whole hot path on one batch: evisel_probe_attention (block-sparse
GQA attention + split-KV merge, text-logit spill) and evisel_evidence_reduce
(token / frame / head maps and A_qf). The headline workload is the 65,664-token
probe (1024 frames x 64 pooled tokens + 128 text tokens, 28 query / 4 KV heads,
d = 128, 128-token tiles, sink + 16-tile window + 32 random tiles per visual
row tile). Inputs are synthetic (seeded), resident in HBM when the timed region
starts, and larger than L2, so no flush is needed between steps.

The same line carries, under "configs", the step timed the same way on every
workload: the 544-token and 4,160-token probes (L2 flushed before every step),
the 28-layer probe (one step = the probe and the accumulating evidence pass of
all 28 layers, each with its own Q/K/V) and the 8-video packed batch.

Prints one JSON line (rank 0). --impl reference times the float64 oracle on
the host cores instead (bounded sample of the same workload).
"""
from __future__ import annotations

import argparse
import hashlib
import json
import os
import statistics
import subprocess
import sys
import tempfile
import time
from concurrent.futures import ThreadPoolExecutor

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

from paper_2608_05780_gb300 import workloads as wl  # noqa: E402

METRIC = "probe-attention TFLOP/s (unmasked) & % GB300 BF16 peak; evidence-map GB/s"


def _env_int(name, default):
    try:
        return int(os.environ.get(name, default))
    except ValueError:
        return default


def workload_stats(probe):
    """Algorithmic work of one probe layer (kept tiles only, full-tile convention)."""
    cfg = probe.cfg
    T, d, hq = cfg.tile, cfg.head_dim, cfg.hq
    elems = 0
    valid = 0
    tiles = 0
    r = 0
    for b in range(len(probe.n_vis)):
        nv = int(probe.n_vis[b])
        nt = int(probe.n_text[b])
        n_vt, n_tt = -(-nv // T), -(-nt // T)
        tl = lambda c, n: min(T, n - c * T)
        for t in range(n_vt):
            rows = tl(t, nv)
            for c in probe.col_idx[probe.row_ptr[r]:probe.row_ptr[r + 1]]:
                cols = tl(int(c), nv)
                elems += rows * cols
                valid += rows * cols if c != t else rows * (rows + 1) // 2
                tiles += 1
            r += 1
        for t in range(n_tt):
            rows = tl(t, nt)
            for c in range(n_vt):
                elems += rows * tl(c, nv); valid += rows * tl(c, nv); tiles += 1
            for u in range(t + 1):
                cols = tl(u, nt)
                elems += rows * cols
                valid += rows * cols if u != t else rows * (rows + 1) // 2
                tiles += 1
    flop = 4.0 * d * hq * elems
    flop_valid = 4.0 * d * hq * valid
    n_tok = int(probe.cu_seqlens[-1])
    spill = sum(hq * int(nt) * int(nv) * 4 for nv, nt in zip(probe.n_vis, probe.n_text))
    lse_read = sum(hq * int(nt) * 4 for nt in probe.n_text)
    total_vis = int(np.sum(probe.n_vis))
    frames = total_vis // cfg.tokens_per_frame
    maps = 4 * (hq * total_vis + hq * frames + len(probe.n_vis) * hq + frames)
    return dict(flop=flop, flop_valid=flop_valid, tiles=tiles, n_tok=n_tok, spill_bytes=spill,
                evidence_bytes=spill + lse_read + maps, map_bytes=maps)


def _peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        j = json.load(open(p))
        return dict(hbm=j["hbm_gbs"], bf16=j["bf16_tflops"], bf16_sus=j["bf16_tflops_sustained"],
                    sm_max=j.get("sm_max_mhz"), source="measured")
    return dict(hbm=6800.0, bf16=1900.0, bf16_sus=1700.0, sm_max=2070.0, source="fallback")


def _kernel_sha():
    h = hashlib.sha256()
    for f in ("probe_attn.cu", "sm103_ptx.cuh", "evisel_internal.h"):
        h.update(open(os.path.join(ROOT, "paper_2608_05780_gb300", "csrc", f), "rb").read())
    return h.hexdigest()[:16]


def _traffic(workload):
    """DRAM bytes per launch of the attention kernel from the committed ncu summary, if current."""
    path = os.path.join(ROOT, "profiles", "probe_attn_long65k_traffic.txt")
    if not os.path.exists(path):
        return None
    kv = {}
    for line in open(path):
        if ":" in line and not line.startswith("#"):
            k, v = line.split(":", 1)
            kv[k.strip()] = v.strip()
    if kv.get("source_sha") != _kernel_sha() or kv.get("workload") != workload:
        return None
    try:
        return float(kv["dram_bytes_per_launch"])
    except (KeyError, ValueError):
        return None


class ClockSampler:
    """nvidia-smi sampling of SM clocks and throttle reasons during the timed region."""
    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, index):
        self.index = index
        self.proc = None
        self.file = None

    def start(self):
        try:
            self.file = tempfile.NamedTemporaryFile("w+", suffix=".csv", delete=False)
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.index), f"--query-gpu={self.FIELDS}", "--format=csv,noheader,nounits",
                 "-lms", "100"], stdout=self.file, stderr=subprocess.DEVNULL)
        except (OSError, FileNotFoundError):
            self.proc = None

    def stop(self):
        if self.proc is None:
            return None
        time.sleep(0.25)
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
        self.file.flush()
        self.file.seek(0)
        rows = [r.split(",") for r in self.file.read().strip().splitlines() if r.count(",") >= 8]
        os.unlink(self.file.name)
        if not rows:
            return None
        sm = [float(r[1]) for r in rows if r[1].strip().replace(".", "").isdigit()]
        smax = [float(r[2]) for r in rows if r[2].strip().replace(".", "").isdigit()]
        pw = [float(r[3]) for r in rows if r[3].strip().replace(".", "").isdigit()]
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({names[i] for r in rows for i in range(4) if r[5 + i].strip() == "Active"})
        return {"sm_mhz": statistics.median(sm) if sm else None, "sm_max_mhz": max(smax) if smax else None,
                "sm_mhz_min": min(sm) if sm else None, "power_w_max": max(pw) if pw else None,
                "reasons": reasons, "samples": len(rows)}


def _oracle_sample(probe, max_rows):
    """Rows of the longest visual row tiles plus the text rows: a bounded slice of the workload."""
    cfg = probe.cfg
    T = cfg.tile
    counts = np.diff(probe.row_ptr)
    order = np.argsort(-counts, kind="stable")
    rows, flop = [], 0.0
    s0, nv = int(probe.cu_seqlens[0]), int(probe.n_vis[0])
    nt = int(probe.n_text[0])
    text_rows = list(range(s0 + nv, s0 + nv + nt))
    n_vt = -(-nv // T)
    rows += text_rows
    flop += 4.0 * cfg.head_dim * cfg.hq * nt * (nv + -(-nt // T) * T)
    for r in order:
        if len(rows) >= max_rows or r >= n_vt:
            break
        rl = min(T, nv - int(r) * T)
        rows += list(range(s0 + int(r) * T, s0 + int(r) * T + rl))
        flop += 4.0 * cfg.head_dim * cfg.hq * rl * int(counts[r]) * T
    return np.array(rows), flop


def run_oracle(probe, max_rows):
    import oracle
    rows, flop = _oracle_sample(probe, max_rows)
    t0 = time.perf_counter()
    oracle.probe_rows(probe.q, probe.k, probe.v, probe.cu_seqlens, probe.n_vis, probe.cfg.tile, probe.row_ptr,
                      probe.col_idx, rows)
    oracle.evidence(probe.q, probe.k, probe.cu_seqlens, probe.n_vis, probe.cfg.tokens_per_frame)
    dt = time.perf_counter() - t0
    return flop, dt, len(rows)


def bench_reference(args, cfg):
    rank = _env_int("RANK", 0)
    if rank != 0:
        return 0
    probe = wl.make_probe(cfg)
    st = workload_stats(probe)
    for _ in range(args.warmup):
        run_oracle(probe, args.ref_rows)
    flops, times, nrows = 0.0, 0.0, 0
    for _ in range(args.steps):
        f, dt, nrows = run_oracle(probe, args.ref_rows)
        flops += f
        times += dt
    value = flops / times / 1e12
    cores = os.cpu_count()
    sample = (f"{nrows} query rows (the text rows plus the longest visual row tiles) of {cfg.name}, all "
              f"{cfg.hq} heads, dense float64 rows, plus the full text-row evidence maps; FLOP counted "
              f"over the rows' kept tiles")
    line = {"impl": "reference", "metric": METRIC, "value": value, "unit": "TFLOP/s", "n_gpus": args.gpus,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": 1e3 * times / args.steps,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
            "data": "synthetic", "config": _config_dict(cfg, st),
            "cpu_baseline": {"value": value, "unit": "TFLOP/s", "cores": cores, "kind": "oracle",
                             "sample": sample},
            "e2e": {"value": value, "unit": "TFLOP/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)
    return 0


def _max_over_ranks(x, world):
    """x at one rank; else the largest x over the ranks (the slowest rank's
    time), by an all-reduce on the process group's device (CUDA under NCCL,
    the host under gloo)."""
    if world <= 1:
        return float(x)
    import torch
    import torch.distributed as dist
    dev = "cuda" if dist.get_backend() == "nccl" else "cpu"
    t = torch.tensor([float(x)], dtype=torch.float64, device=dev)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def _whole_job_tflops(world, flop_per_replica_step, ms_per_step):
    """Whole-job throughput: one step's FLOP on every replica over the
    (max-over-ranks) step time."""
    return world * flop_per_replica_step / (ms_per_step * 1e-3) / 1e12


def _config_dict(cfg, st):
    return {"workload": f"{cfg.name}: {cfg.description}", "tokens": st["n_tok"], "kept_tiles": st["tiles"],
            "layers": cfg.layers, "videos": cfg.num_videos, "hq": cfg.hq, "hkv": cfg.hkv,
            "head_dim": cfg.head_dim, "tile": cfg.tile, "tokens_per_frame": cfg.tokens_per_frame,
            "l2": "inputs larger than L2 (no flush)", "parallelism": "replicas"}


L2_FLUSH_BYTES = 256 * 1024 * 1024     # twice the GB300's L2


def _gpu_local_cpus(device_index):
    """Host CPUs on the NUMA node of the GPU's PCI device (empty if unknown):
    pinned host buffers first touched from these CPUs sit in the memory
    nearest to the GPU, and copies from them take the shortest path."""
    import torch
    try:
        p = torch.cuda.get_device_properties(device_index)
        bus = f"{p.pci_domain_id:04x}:{p.pci_bus_id:02x}:{p.pci_device_id:02x}.0"
        with open(f"/sys/bus/pci/devices/{bus}/local_cpulist") as fh:
            spec = fh.read().strip()
    except (AttributeError, OSError, ValueError):
        return set()
    cpus = set()
    for part in spec.split(","):
        if part:
            a, _, b = part.partition("-")
            cpus |= set(range(int(a), int(b or a) + 1))
    return cpus & os.sched_getaffinity(0)


def bench_config(ev, name, args, peaks):
    """The step (probe + evidence over every layer) of one workload, timed on
    the launch stream with CUDA events: the whole step, and per layer the
    probe call and the evidence call, once through each evidence path (the
    text-row logit spill read back by the HBM-bound reduce, and the
    recompute pass without the spill). Workloads whose inputs fit in L2 get a
    256 MB write before every timed step (outside the timed interval)."""
    import torch
    cfg = wl.CONFIGS[name]
    layers = cfg.layers
    if layers > 1:
        mask = wl.build_mask(cfg)
        with ThreadPoolExecutor(max(1, min(8, os.cpu_count() or 1))) as ex:
            probes = list(ex.map(lambda l: wl.make_probe(cfg, l, mask=mask), range(layers)))
    else:
        probes = [wl.make_probe(cfg)]
    probe = probes[0]
    st = workload_stats(probe)                  # per layer: every layer has the same shapes and mask
    dev = []
    for p in probes:
        dev.append(tuple(torch.from_numpy(x).cuda().to(torch.bfloat16) for x in (p.q, p.k, p.v)))
    del probes
    q0 = dev[0][0]
    n, hq, d = q0.shape
    in_bytes = layers * sum(t.numel() * t.element_size() for t in dev[0])
    flush = in_bytes + st["spill_bytes"] < 4 * L2_FLUSH_BYTES
    flush_buf = torch.empty(L2_FLUSH_BYTES // 4, dtype=torch.float32, device="cuda") if flush else None
    o = torch.empty_like(q0)
    lse = torch.empty((hq, n), dtype=torch.float32, device="cuda")
    total_vis = int(np.sum(probe.n_vis))
    frames = total_vis // cfg.tokens_per_frame
    maps = [torch.zeros((hq, total_vis), device="cuda"), torch.zeros((hq, frames), device="cuda"),
            torch.zeros((len(probe.n_vis), hq), device="cuda"), torch.zeros((frames,), device="cuda")]
    stream = torch.cuda.current_stream()
    ev_t = lambda: torch.cuda.Event(enable_timing=True)

    def timed_steps(text_evidence):
        """(step ms, probe ms, evidence ms) averaged over args.steps steps of one evidence path."""
        ws = ev.Workspace()

        def step(marks=None):
            for layer, (q, k, v) in enumerate(dev):
                if marks:
                    marks[layer][0].record(stream)
                ev.evisel_probe_attention(q, k, v, probe.cu_seqlens, probe.n_vis, cfg.tokens_per_frame, cfg.tile,
                                          probe.row_ptr, probe.col_idx, ws=ws, o=o, lse=lse,
                                          text_evidence=text_evidence)
                if marks:
                    marks[layer][1].record(stream)
                ev.evisel_evidence_reduce(ws, hq, probe.n_vis, cfg.tokens_per_frame, len(probe.n_vis), tok=maps[0],
                                          frame=maps[1], head=maps[2], aqf=maps[3], accumulate=layer > 0)
                if marks:
                    marks[layer][2].record(stream)

        for _ in range(args.warmup):
            step()
        torch.cuda.synchronize()
        if ev.evisel_status(ws) != 0:
            raise RuntimeError(f"{name}: device status reported an error")
        bounds = [(ev_t(), ev_t()) for _ in range(args.steps)]
        marks = [[[ev_t() for _ in range(3)] for _ in range(layers)] for _ in range(args.steps)]
        for i in range(args.steps):
            if flush_buf is not None:
                flush_buf.zero_()
            bounds[i][0].record(stream)
            step(marks[i])
            bounds[i][1].record(stream)
        torch.cuda.synchronize()
        status = ev.evisel_status(ws)
        ws_bytes = ws.nbytes
        ws.free()
        if status != 0:
            raise RuntimeError(f"{name}: device status reported an error")
        if not all(bool(torch.isfinite(m).all()) for m in maps):
            raise RuntimeError(f"{name}: non-finite evidence maps")
        step_ms = sum(a.elapsed_time(b) for a, b in bounds) / args.steps
        attn_ms = sum(m[0].elapsed_time(m[1]) for s_ in marks for m in s_) / args.steps
        ev_ms = sum(m[1].elapsed_time(m[2]) for s_ in marks for m in s_) / args.steps
        return step_ms, attn_ms, ev_ms, ws_bytes

    step_ms, attn_ms, ev_ms, _ = timed_steps(False)
    rc_step_ms, rc_attn_ms, rc_ev_ms, rc_ws = timed_steps(True)
    flop = layers * st["flop"]
    attn_tflops = flop / (attn_ms * 1e-3) / 1e12
    ev_gbs = layers * st["evidence_bytes"] / (ev_ms * 1e-3) / 1e9
    rc_attn_tflops = flop / (rc_attn_ms * 1e-3) / 1e12
    return {"workload": f"{cfg.name}: {cfg.description}", "tokens": st["n_tok"], "layers": layers,
            "videos": cfg.num_videos, "kept_tiles_per_layer": st["tiles"], "flop_per_step": flop,
            "step_ms": step_ms, "tflops": flop / (step_ms * 1e-3) / 1e12,
            "tokens_per_s": st["n_tok"] * layers / (step_ms * 1e-3),
            "attention_ms": attn_ms, "attention_tflops": attn_tflops,
            "attention_frac_of_bf16_peak": attn_tflops / peaks["bf16"],
            "attention_ms_at_60pct_of_peak": flop / (0.6 * peaks["bf16"] * 1e12) * 1e3,
            "evidence_ms": ev_ms, "evidence_bytes": layers * st["evidence_bytes"], "evidence_gbs": ev_gbs,
            "evidence_frac_of_hbm": ev_gbs / peaks["hbm"],
            "recompute_evidence": {
                "note": "the same step with text_evidence = 1: the probe writes no text-row logit spill and the "
                        "evidence call forms the text-row probabilities from q, k and the saved LSE",
                "step_ms": rc_step_ms, "tflops": flop / (rc_step_ms * 1e-3) / 1e12,
                "tokens_per_s": st["n_tok"] * layers / (rc_step_ms * 1e-3),
                "attention_ms": rc_attn_ms, "attention_tflops": rc_attn_tflops,
                "attention_frac_of_bf16_peak": rc_attn_tflops / peaks["bf16"],
                "evidence_ms": rc_ev_ms, "workspace_bytes": rc_ws},
            "l2": "256 MB write before every step (untimed)" if flush else "inputs larger than L2 (no flush)"}


def bench_topp_sparse(ev, args, peaks):
    """The top-p path (Appendix Eq. 6-9, blocks of N_v tokens, tau_p = 0.97)
    where retention keeps a small share of each row's history: the 65K probe
    with concentrated attention (long65k_sparse). Times the builder, the probe
    on the tile union with the per-row bits, and, for comparison, the probe on
    the same inputs under the static mask; the kept share is counted on a
    sample of rows from the builder's own bits."""
    import torch
    cfg = wl.CONFIGS["long65k_sparse"]
    probe = wl.make_probe(cfg)
    st = workload_stats(probe)
    q, k, v = (torch.from_numpy(x).cuda().to(torch.bfloat16) for x in (probe.q, probe.k, probe.v))
    n, hq, d = q.shape
    npf, tau = cfg.tokens_per_frame, 0.97
    o = torch.empty_like(q)
    lse = torch.empty((hq, n), dtype=torch.float32, device="cuda")
    stream = torch.cuda.current_stream()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)

    def timed(fn):
        for _ in range(max(1, args.warmup)):
            fn()
        torch.cuda.synchronize()
        e0.record(stream)
        for _ in range(args.steps):
            fn()
        e1.record(stream)
        torch.cuda.synchronize()
        return e0.elapsed_time(e1) / args.steps

    ws = ev.Workspace()
    keep, uni, ws = ev.evisel_topp_mask(q, k, probe.cu_seqlens, probe.n_vis, npf, cfg.tile, npf, tau, ws=ws)
    build_ms = timed(lambda: ev.evisel_topp_mask(q, k, probe.cu_seqlens, probe.n_vis, npf, cfg.tile, npf, tau,
                                                 ws=ws))
    row_ptr, col_idx = ev.tile_union_to_csr(uni, probe.n_vis, cfg.tile)
    uargs = (q, k, v, probe.cu_seqlens, probe.n_vis, npf, cfg.tile, row_ptr, col_idx)
    ws_p = ev.Workspace()
    union_ms = timed(lambda: ev.evisel_probe_attention(*uargs, ws=ws_p, o=o, lse=lse, keep=keep, keep_block=npf))
    sargs = (q, k, v, probe.cu_seqlens, probe.n_vis, npf, cfg.tile, probe.row_ptr, probe.col_idx)
    ws_s = ev.Workspace()
    static_ms = timed(lambda: ev.evisel_probe_attention(*sargs, ws=ws_s, o=o, lse=lse))
    status = [ev.evisel_status(w) for w in (ws, ws_p, ws_s)]
    # kept share on sampled rows: retained blocks (own block excluded) over |H_i|
    rows = np.random.default_rng(0).integers(0, n, 256)
    bits = keep[:, :, torch.as_tensor(rows, device="cuda")].cpu().numpy().view(np.uint32)   # [hq, words, rows]
    bits = np.ascontiguousarray(bits.transpose(0, 2, 1))                                       # [hq, rows, words]
    kept = np.unpackbits(bits.view(np.uint8), axis=2).sum(axis=2).astype(np.int64) - 1         # own block excluded
    nv = int(probe.n_vis[0])
    hist = np.where(rows < nv, rows // npf, nv // npf + (rows - nv) // npf)
    share = (kept / np.maximum(hist, 1)[None, :])[:, hist >= 64]
    for w in (ws, ws_p, ws_s):
        w.free()
    if any(status):
        raise RuntimeError("device status reported an error")
    # union work in the attention's convention: every kept (row tile, kv tile) pair, full tiles, plus text rows
    ust = workload_stats(wl.Probe(cfg, 0, probe.q[:0], probe.k[:0], probe.v[:0], probe.cu_seqlens, probe.n_vis,
                                  row_ptr, col_idx, probe.planted))
    return {"workload": f"{cfg.name}: {cfg.description}", "block": npf, "tau_p": tau,
            "builder_ms": build_ms,
            "kept_share_of_history": {"median": float(np.median(share)), "mean": float(np.mean(share)),
                                      "sampled_rows": int(share.shape[1]), "heads": hq},
            "union_tiles": int(row_ptr[-1]), "static_mask_tiles": int(probe.row_ptr[-1]),
            "probe_on_union_ms": union_ms, "probe_on_union_tflops": ust["flop"] / (union_ms * 1e-3) / 1e12,
            "probe_on_union_frac_of_bf16_peak": ust["flop"] / (union_ms * 1e-3) / 1e12 / peaks["bf16"],
            "probe_static_mask_ms": static_ms,
            "builder_plus_union_probe_ms": build_ms + union_ms}


def bench_ours(args, cfg):
    import torch
    import torch.distributed as dist

    import paper_2608_05780_gb300 as ev

    world = _env_int("WORLD_SIZE", 1)
    rank = _env_int("RANK", 0)
    local = _env_int("LOCAL_RANK", 0)
    if world > 1:
        dist.init_process_group("nccl")
    torch.cuda.set_device(local)
    ev.ensure_built()
    probe = wl.make_probe(cfg)
    st = workload_stats(probe)
    q = torch.from_numpy(probe.q).cuda().to(torch.bfloat16)
    k = torch.from_numpy(probe.k).cuda().to(torch.bfloat16)
    v = torch.from_numpy(probe.v).cuda().to(torch.bfloat16)
    n, hq, d = q.shape
    o = torch.empty_like(q)
    lse = torch.empty((hq, n), dtype=torch.float32, device="cuda")
    total_vis = int(np.sum(probe.n_vis))
    frames = total_vis // cfg.tokens_per_frame
    maps = [torch.zeros((hq, total_vis), device="cuda"), torch.zeros((hq, frames), device="cuda"),
            torch.zeros((len(probe.n_vis), hq), device="cuda"), torch.zeros((frames,), device="cuda")]
    ws = ev.Workspace()
    stream = torch.cuda.current_stream()

    def step(ev_marks=None):
        if ev_marks:
            ev_marks[0].record(stream)
        ev.evisel_probe_attention(q, k, v, probe.cu_seqlens, probe.n_vis, cfg.tokens_per_frame, cfg.tile,
                                  probe.row_ptr, probe.col_idx, ws=ws, o=o, lse=lse)
        if ev_marks:
            ev_marks[1].record(stream)
        ev.evisel_evidence_reduce(ws, hq, probe.n_vis, cfg.tokens_per_frame, len(probe.n_vis), tok=maps[0],
                                  frame=maps[1], head=maps[2], aqf=maps[3])
        if ev_marks:
            ev_marks[2].record(stream)

    for _ in range(args.warmup):
        step()
    torch.cuda.synchronize()
    if ev.evisel_status(ws) != 0:
        raise RuntimeError("device status reported an error")

    marks = [[torch.cuda.Event(enable_timing=True) for _ in range(3)] for _ in range(args.steps)]
    clocks = ClockSampler(local)
    if world > 1:
        dist.barrier()
    torch.cuda.synchronize()
    clocks.start()
    t_start = torch.cuda.Event(enable_timing=True)
    t_end = torch.cuda.Event(enable_timing=True)
    t_start.record(stream)
    for i in range(args.steps):
        step(marks[i])
    t_end.record(stream)
    torch.cuda.synchronize()
    clk = clocks.stop()
    if world > 1:
        dist.barrier()
    elapsed_ms = t_start.elapsed_time(t_end)
    attn_ms = [m[0].elapsed_time(m[1]) for m in marks]
    ev_ms = [m[1].elapsed_time(m[2]) for m in marks]
    elapsed_ms = _max_over_ranks(elapsed_ms, world)
    ms_step = elapsed_ms / args.steps
    value = _whole_job_tflops(world, st["flop"], ms_step)
    attn_avg = sum(attn_ms) / len(attn_ms)
    ev_avg = sum(ev_ms) / len(ev_ms)
    peaks = _peaks()
    attn_tflops = st["flop"] / (attn_avg * 1e-3) / 1e12
    ev_gbs = st["evidence_bytes"] / (ev_avg * 1e-3) / 1e9

    # End to end through the public API with host buffers: every step copies its
    # inputs in from pinned host memory and its evidence maps out. The copies run
    # on a second stream into a second set of device buffers, so that the inputs
    # of step i + 1 and the maps of step i move while step i computes (the
    # first step's inputs and the last step's maps are inside the timed region).
    # Host buffers on the GPU's NUMA node: the process runs on the GPU's local
    # CPUs from here on, so that the pinned buffers are first touched there.
    local_cpus = _gpu_local_cpus(local)
    if local_cpus:
        os.sched_setaffinity(0, local_cpus)
    hq_, hk_, hv_ = (t.cpu().pin_memory() for t in (q, k, v))
    host_maps = [m.cpu().pin_memory() for m in maps]
    h2d = sum(t.numel() * t.element_size() for t in (hq_, hk_, hv_))
    d2h = sum(m.numel() * m.element_size() for m in maps)
    copy_stream = torch.cuda.Stream()
    bufs = [(q, k, v), tuple(torch.empty_like(t) for t in (q, k, v))]
    map_bufs = [maps, [torch.empty_like(m) for m in maps]]
    in_ready = [torch.cuda.Event() for _ in range(2)]
    comp_done = [torch.cuda.Event() for _ in range(2)]
    out_done = [torch.cuda.Event() for _ in range(2)]

    def load_inputs(slot):
        with torch.cuda.stream(copy_stream):
            for dst, src in zip(bufs[slot], (hq_, hk_, hv_)):
                dst.copy_(src, non_blocking=True)
            in_ready[slot].record(copy_stream)

    def e2e_run(n_steps, start_evt=None):
        if start_evt is not None:
            copy_stream.wait_event(start_evt)
        load_inputs(0)
        for i in range(n_steps):
            s_ = i % 2
            if i + 1 < n_steps:
                if i >= 1:
                    copy_stream.wait_event(comp_done[(i + 1) % 2])     # buffer free: step i - 1 done
                load_inputs((i + 1) % 2)
            stream.wait_event(in_ready[s_])
            if i >= 2:
                stream.wait_event(out_done[s_])                        # maps of step i - 2 read out
            qi, ki, vi = bufs[s_]
            mi = map_bufs[s_]
            ev.evisel_probe_attention(qi, ki, vi, probe.cu_seqlens, probe.n_vis, cfg.tokens_per_frame, cfg.tile,
                                      probe.row_ptr, probe.col_idx, ws=ws, o=o, lse=lse)
            ev.evisel_evidence_reduce(ws, hq, probe.n_vis, cfg.tokens_per_frame, len(probe.n_vis), tok=mi[0],
                                      frame=mi[1], head=mi[2], aqf=mi[3])
            comp_done[s_].record(stream)
            with torch.cuda.stream(copy_stream):
                copy_stream.wait_event(comp_done[s_])
                for hm, m in zip(host_maps, mi):
                    hm.copy_(m, non_blocking=True)
                out_done[s_].record(copy_stream)
        stream.wait_event(out_done[(n_steps - 1) % 2])

    e2e_run(max(1, args.warmup))
    torch.cuda.synchronize()
    if world > 1:
        dist.barrier()
    e0 = torch.cuda.Event(enable_timing=True)
    e1 = torch.cuda.Event(enable_timing=True)
    e2e_clocks = ClockSampler(local)
    e2e_clocks.start()
    e0.record(stream)
    e2e_run(args.steps, start_evt=e0)
    e1.record(stream)
    torch.cuda.synchronize()
    e2e_clk = e2e_clocks.stop()
    e2e_ms = _max_over_ranks(e0.elapsed_time(e1) / args.steps, world)
    # the copies are done: the last step's maps are on the host
    if not all(np.isfinite(hm.numpy()).all() for hm in host_maps):
        raise RuntimeError("non-finite evidence maps")

    # The copies alone, on the copy stream: what bounds the pipelined loop
    # when they take longer than the step.
    def copy_ms(fn):
        c0, c1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        for _ in range(2):
            fn()
        torch.cuda.synchronize()
        c0.record(copy_stream)
        for _ in range(args.steps):
            fn()
        c1.record(copy_stream)
        torch.cuda.synchronize()
        return c0.elapsed_time(c1) / args.steps

    def h2d_only():
        with torch.cuda.stream(copy_stream):
            for dst, src in zip(bufs[1], (hq_, hk_, hv_)):
                dst.copy_(src, non_blocking=True)

    def d2h_only():
        with torch.cuda.stream(copy_stream):
            for hm, m in zip(host_maps, map_bufs[1]):
                hm.copy_(m, non_blocking=True)

    h2d_ms = copy_ms(h2d_only)
    d2h_ms = copy_ms(d2h_only)
    del bufs[1], map_bufs[1]

    # The intra-frame cue A_if (a row beyond the probe step), timed on its own
    # after the probe whose LSE it reads: HBM-bound (Q, K and LSE of the visual
    # rows in, A_if out), with the diagonal logits recomputed on the tensor cores.
    npf = cfg.tokens_per_frame
    aif = torch.zeros((frames, npf, npf), device="cuda")

    def intra_frame():
        ev.evisel_intra_frame_evidence(q, k, v, probe.cu_seqlens, probe.n_vis, npf, cfg.tile, probe.row_ptr,
                                       probe.col_idx, o, lse, ws, aif=aif)

    for _ in range(max(1, args.warmup)):
        intra_frame()
    torch.cuda.synchronize()
    e0.record(stream)
    for _ in range(args.steps):
        intra_frame()
    e1.record(stream)
    torch.cuda.synchronize()
    if_ms = e0.elapsed_time(e1) / args.steps
    if_bytes = total_vis * (hq * d * 2 + k.shape[1] * d * 2 + hq * 4) + frames * npf * npf * 4
    if_flop = 2.0 * d * 128 * 128 * hq * sum(-(-int(nv) // 128) for nv in probe.n_vis)
    status = ev.evisel_status(ws)
    ws.free()
    if status != 0:
        raise RuntimeError("device status reported an error")

    # The cross-frame cue A_ff / E_ff (a row beyond the probe step): the probe
    # run with its cross-frame partials (an extra output of the attention
    # kernel), then the HBM-bound reduction of those partials, each timed on
    # its own.
    ws_cf = ev.Workspace()
    pargs = (q, k, v, probe.cu_seqlens, probe.n_vis, npf, cfg.tile, probe.row_ptr, probe.col_idx)
    o_cf, lse_cf, ws_cf = ev.evisel_probe_attention(*pargs, ws=ws_cf, cross_frame=True)
    t_frames = np.asarray(probe.n_vis) // npf
    aff = torch.empty(int(np.sum(np.maximum(t_frames - 1, 0) ** 2)), device="cuda")
    eff = torch.empty(frames, device="cuda")

    def probe_cf():
        ev.evisel_probe_attention(*pargs, ws=ws_cf, o=o_cf, lse=lse_cf, cross_frame=True)

    def cross_frame():
        ev.evisel_cross_frame_evidence(*pargs, o_cf, lse_cf, ws_cf, aff=aff, eff=eff)

    def _time(fn):
        for _ in range(max(1, args.warmup)):
            fn()
        torch.cuda.synchronize()
        e0.record(stream)
        for _ in range(args.steps):
            fn()
        e1.record(stream)
        torch.cuda.synchronize()
        return e0.elapsed_time(e1) / args.steps

    pcf_ms = _time(probe_cf)
    cf_ms = _time(cross_frame)
    nnz = int(probe.row_ptr[-1])
    fspill_bytes = hq * nnz * (cfg.tile // npf) * cfg.tile * 4
    cf_bytes = fspill_bytes + hq * total_vis * 4 + aff.numel() * 4 + frames * 4
    status = ev.evisel_status(ws_cf)
    ws_cf.free()
    if status != 0:
        raise RuntimeError("device status reported an error")

    # The step with the recompute evidence pass (text_evidence = 1): the probe
    # without the text-row logit spill, then the evidence formed from Q, K and
    # the LSE on the tensor cores. Same outputs; timed like the step.
    ws_te = ev.Workspace()
    maps_te = [torch.zeros_like(m) for m in maps]
    ev.evisel_probe_attention(*pargs, ws=ws_te, o=o_cf, lse=lse_cf, text_evidence=True)

    def probe_te():
        ev.evisel_probe_attention(*pargs, ws=ws_te, o=o_cf, lse=lse_cf, text_evidence=True)

    def evid_te():
        ev.evisel_evidence_reduce(ws_te, hq, probe.n_vis, npf, len(probe.n_vis), tok=maps_te[0],
                                  frame=maps_te[1], head=maps_te[2], aqf=maps_te[3])

    def step_te():
        probe_te()
        evid_te()

    te_step_ms = _time(step_te)

    # The top-p block retention of the sparse prefill (Appendix Eq. 6-9) on the
    # same inputs, blocks of N_v tokens, tau_p = 0.97 (outside the step: the
    # workloads' masks are static).
    ws_tp = ev.Workspace()
    keep_tp, uni_tp, ws_tp = ev.evisel_topp_mask(q, k, probe.cu_seqlens, probe.n_vis, npf, cfg.tile, npf, 0.97,
                                                 ws=ws_tp)

    def topp():
        ev.evisel_topp_mask(q, k, probe.cu_seqlens, probe.n_vis, npf, cfg.tile, npf, 0.97, ws=ws_tp)

    tp_ms = _time(topp)
    # the probe restricted to each row's retained blocks: the row tiles' union
    # as the tile mask, the per-row bits inside
    tp_row_ptr, tp_col_idx = ev.tile_union_to_csr(uni_tp, probe.n_vis, cfg.tile)
    tp_args = (q, k, v, probe.cu_seqlens, probe.n_vis, npf, cfg.tile, tp_row_ptr, tp_col_idx)

    def probe_topp():
        ev.evisel_probe_attention(*tp_args, ws=ws_tp, o=o_cf, lse=lse_cf, keep=keep_tp, keep_block=npf)

    tpp_ms = _time(probe_topp)
    tp_tiles = int(tp_row_ptr[-1])
    # the evidence of the coarse token-level map (Eq. 10-11) on the same sets
    ev.evisel_topp_mask(q, k, probe.cu_seqlens, probe.n_vis, npf, cfg.tile, npf, 0.97, ws=ws_tp)
    maps_co = [torch.empty_like(m) for m in maps]

    def coarse():
        ev.evisel_coarse_evidence(q, k, probe.cu_seqlens, probe.n_vis, npf, cfg.tile, npf, keep_tp, ws_tp,
                                  tok=maps_co[0], frame=maps_co[1], head=maps_co[2], aqf=maps_co[3])

    co_ms = _time(coarse)
    status = ev.evisel_status(ws_tp)
    ws_tp.free()
    del keep_tp, uni_tp
    if status != 0:
        raise RuntimeError("device status reported an error")
    n_blk = int(sum(int(nv) // npf + -(-int(nt) // npf) for nv, nt in zip(probe.n_vis, probe.n_text)))
    # tensor work of the builder: 6 passes of q k_bar^T over each row's history, head by head
    tp_flop = 6 * 2.0 * d * hq * sum(
        sum((p_ // npf) for p_ in range(int(nv))) + sum(int(nv) // npf + t // npf for t in range(int(nt)))
        for nv, nt in zip(probe.n_vis, probe.n_text))
    te_probe_ms = _time(probe_te)
    te_ev_ms = _time(evid_te)
    status = ev.evisel_status(ws_te)
    te_ws_bytes = ws_te.nbytes
    ws_te.free()
    if status != 0:
        raise RuntimeError("device status reported an error")

    topp_sparse = None if args.no_configs else bench_topp_sparse(ev, args, peaks)
    torch.cuda.empty_cache()

    # Every workload's step, timed the same way (replicas: each rank times its own).
    configs = {}
    if not args.no_configs:
        cclk = ClockSampler(local)
        cclk.start()
        for name in ("tiny", "single", "depth28", "varlen8"):
            configs[name] = bench_config(ev, name, args, peaks)
            torch.cuda.empty_cache()
        configs["clocks"] = cclk.stop()
    configs["long65k"] = {"workload": f"{cfg.name}: {cfg.description}", "tokens": st["n_tok"], "layers": 1,
                          "videos": cfg.num_videos, "kept_tiles_per_layer": st["tiles"], "flop_per_step": st["flop"],
                          "step_ms": ms_step, "tflops": st["flop"] / (ms_step * 1e-3) / 1e12,
                          "tokens_per_s": st["n_tok"] / (ms_step * 1e-3),
                          "attention_ms": attn_avg, "attention_tflops": attn_tflops,
                          "attention_frac_of_bf16_peak": attn_tflops / peaks["bf16"],
                          "attention_ms_at_60pct_of_peak": st["flop"] / (0.6 * peaks["bf16"] * 1e12) * 1e3,
                          "evidence_ms": ev_avg, "evidence_bytes": st["evidence_bytes"], "evidence_gbs": ev_gbs,
                          "evidence_frac_of_hbm": ev_gbs / peaks["hbm"], "l2": "inputs larger than L2 (no flush)",
                          "recompute_evidence": {
                              "note": "text_evidence_recompute above: the step without the text-row logit spill",
                              "step_ms": te_step_ms, "tflops": st["flop"] / (te_step_ms * 1e-3) / 1e12,
                              "tokens_per_s": st["n_tok"] / (te_step_ms * 1e-3),
                              "attention_ms": te_probe_ms,
                              "attention_tflops": st["flop"] / (te_probe_ms * 1e-3) / 1e12,
                              "attention_frac_of_bf16_peak": st["flop"] / (te_probe_ms * 1e-3) / 1e12 / peaks["bf16"],
                              "evidence_ms": te_ev_ms, "workspace_bytes": te_ws_bytes},
                          "note": "the headline step (value, attention, evidence above)"}

    line = None
    if rank == 0:
        line = {"metric": METRIC, "value": value, "unit": "TFLOP/s", "n_gpus": world, "steps": args.steps,
                "warmup": args.warmup, "ms_per_step": ms_step, "higher_is_better": True, "scaling": "weak",
                "vs_baseline": None, "dtype": "bf16", "data": "synthetic", "config": _config_dict(cfg, st),
                "frac_of_bf16_peak": value / world / peaks["bf16"],
                "tokens_per_s": world * st["n_tok"] * cfg.layers / (ms_step * 1e-3),
                "flop_per_step": st["flop"], "flop_causal_valid_per_step": st["flop_valid"],
                "attention": {"ms": attn_avg, "tflops": attn_tflops, "frac_of_bf16_peak": attn_tflops / peaks["bf16"],
                              "frac_of_bf16_sustained": attn_tflops / peaks["bf16_sus"],
                              "tflops_causal_valid": st["flop_valid"] / (attn_avg * 1e-3) / 1e12},
                "evidence": {"ms": ev_avg, "gbs": ev_gbs, "frac_of_hbm": ev_gbs / peaks["hbm"],
                             "bytes": st["evidence_bytes"]},
                "roofline": {"bound": "tensor", "achieved": attn_tflops, "peak": peaks["bf16"], "unit": "TFLOP/s",
                             "frac": attn_tflops / peaks["bf16"],
                             "traffic": _traffic(cfg.name),
                             "kernel": "probe_attn (evisel_probe_attention: probe_attn_kernel + attn_combine)",
                             "peak_source": f"{peaks['source']} bf16 burst"},
                "intra_frame": {"ms": if_ms, "gbs": if_bytes / (if_ms * 1e-3) / 1e9,
                                "frac_of_hbm": if_bytes / (if_ms * 1e-3) / 1e9 / peaks["hbm"], "bytes": if_bytes,
                                "tflops": if_flop / (if_ms * 1e-3) / 1e12},
                "topp_mask": {"ms": tp_ms, "block": npf, "tau_p": 0.97, "blocks": n_blk,
                              "tflops_history": tp_flop / (tp_ms * 1e-3) / 1e12,
                              "probe_ms": tpp_ms, "union_tiles": tp_tiles, "coarse_evidence_ms": co_ms,
                              "static_mask_tiles": int(probe.row_ptr[-1])},
                "text_evidence_recompute": {"step_ms": te_step_ms, "probe_ms": te_probe_ms, "evidence_ms": te_ev_ms,
                                            "tflops": st["flop"] / (te_step_ms * 1e-3) / 1e12,
                                            "workspace_bytes": te_ws_bytes},
                "cross_frame": {"probe_ms": pcf_ms, "probe_partials_bytes": fspill_bytes,
                                "probe_overhead_ms": pcf_ms - attn_avg,
                                "ms": cf_ms, "gbs": cf_bytes / (cf_ms * 1e-3) / 1e9,
                                "frac_of_hbm": cf_bytes / (cf_ms * 1e-3) / 1e9 / peaks["hbm"], "bytes": cf_bytes},
                "e2e": {"value": _whole_job_tflops(world, st["flop"], e2e_ms), "unit": "TFLOP/s",
                        "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h, "ms_per_step": e2e_ms,
                        "h2d_ms_alone": h2d_ms, "h2d_gbs": h2d / (h2d_ms * 1e-3) / 1e9,
                        "d2h_ms_alone": d2h_ms, "d2h_gbs": d2h / (d2h_ms * 1e-3) / 1e9,
                        "host_buffers": (f"pinned, first touched on the GPU's {len(local_cpus)} local CPUs"
                                         if local_cpus else "pinned (GPU NUMA node unknown)"),
                        "pipeline": "inputs of step i+1 and maps of step i copied on a second stream while "
                                    "step i computes",
                        "clocks": e2e_clk},
                "gpu_launches": args.steps * (4 if _has_combine(probe, torch.cuda.get_device_properties(local).multi_processor_count) else 3),
                "clocks": clk,
                "topp_sparse": topp_sparse,
                "configs": configs}
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        flop, dt, nrows = run_oracle(probe, args.ref_rows)
        line["cpu_baseline"] = {"value": flop / dt / 1e12, "unit": "TFLOP/s", "cores": os.cpu_count(),
                                "kind": "oracle",
                                "sample": f"{nrows} query rows (text rows + longest visual row tiles) of "
                                          f"{cfg.name}, all heads, plus the full text-row evidence maps; "
                                          f"{dt:.1f} s"}
    if line is not None:
        print(json.dumps(line), flush=True)
    if world > 1:
        dist.barrier()
        dist.destroy_process_group()
    return 0


def _has_combine(probe, sms):
    """Whether the probe call launches the split-KV combine: some text row tile
    has more kv tiles than the planner's split length (the longest visual row,
    at least 8, raised to half of one SM's share of the tile work, capped at 64)."""
    cfg = probe.cfg
    counts = np.diff(probe.row_ptr)
    blocks = cfg.hkv * -(-(cfg.hq // cfg.hkv) // (2 * (128 // cfg.tile)))
    work = int(counts.sum())
    rows = []
    for nv, nt in zip(probe.n_vis, probe.n_text):
        n_vt, n_tt = -(-int(nv) // cfg.tile), -(-int(nt) // cfg.tile)
        rows += [n_vt + t + 1 for t in range(n_tt)]
    work = (work + sum(rows)) * blocks
    split = max(int(counts.max()) if counts.size else 1, 8, min(64, work // sms // 2))
    return any(r > split for r in rows)


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=20)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--config", default="long65k", choices=sorted(n for n, c in wl.CONFIGS.items() if c.layers == 1),
                    help="workload of the headline step (single-layer workloads; the 28-layer step is "
                         "timed under 'configs')")
    ap.add_argument("--ref-rows", type=int, default=256)
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-configs", action="store_true", help="skip the per-workload steps under 'configs'")
    args = ap.parse_args()
    if args.warmup < 3:
        args.warmup = 3
    cfg = wl.CONFIGS[args.config]
    if args.impl == "reference":
        return bench_reference(args, cfg)
    return bench_ours(args, cfg)


if __name__ == "__main__":
    sys.exit(main())
