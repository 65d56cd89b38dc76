#!/usr/bin/env python3
"""Benchmark of PACE's condense-and-extract hot path on GB300.

One step = the whole hot path on one 4K image per GPU: APC density, APC resample
(target size read on the device), ViT received attention, LLM text->visual attention,
DDAE fusion + top-K, gather of the kept embedding rows.  Inputs are seeded synthetic
arrays shaped like Qwen2.5-VL-7B (3836x2156 image: 42196 patches, ViT Q/K
[42196,16,80] bf16; LLM Q [256,28,128], K [10549,4,128] bf16; embeddings
[10549,3584] bf16; keep 10 % = 1055 tokens).

    python bench.py [--gpus N] [--steps K] [--warmup W] [--impl ours|reference]

Prints one JSON line.  `value` is microseconds per image with inputs resident in HBM,
timed with CUDA events around each step (each libpace call replayed from a CUDA graph),
L2 flushed by a 256 MiB write before every step.  `e2e` is the same metric through the
Python binding with the inputs copied from pinned host memory and the results copied
back inside the timed region (two device input slots, so one image's copies run under the
previous image's calls; `e2e.latency_us_one_image` is one step with nothing else in
flight).  Under torchrun every rank processes its own image
(weak scaling, no collective on the data path); the max over ranks is reported.
`--impl reference` times the fp64 CPU oracle on a bounded sample of the same workload.
"""
from __future__ import annotations

import argparse
import hashlib
import json
import math
import os
import re
import statistics
import subprocess
import sys
import tempfile
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "µs per image for APC+DDAE score/select (4K config); % tensor/HBM peak"
UNIT = "us/image"
WORKLOAD = "img4k"
KEEP = 0.10
FLUSH_BYTES = 256 << 20
FALLBACK_PEAKS = {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0}


# ----------------------------------------------------------------------------------------------
# shared helpers
# ----------------------------------------------------------------------------------------------
def load_peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(path) as f:
            p = json.load(f)
        return p, "measured"
    except (OSError, ValueError):
        return dict(FALLBACK_PEAKS), "fallback"


def profiled_traffic():
    """DRAM bytes per ViT-importance call from the committed ncu summary, or None when the
    kernel source has changed since those counters were taken."""
    path = os.path.join(ROOT, "profiles", "vit_importance_img4k.md")
    src = os.path.join(ROOT, "paper_2608_27206_gb300", "csrc", "attn.cu")
    try:
        text = open(path).read()
        t = re.search(r"traffic_bytes_per_launch:\s*(\d+)", text)
        h = re.search(r"sha256\[:16\]\s*([0-9a-f]{16})", text)
        cur = hashlib.sha256(open(src, "rb").read()).hexdigest()[:16]
        if t and h and h.group(1) == cur:
            return int(t.group(1))
    except OSError:
        pass
    return None


def workload_config(wl, keep):
    s = wl.specs[0]
    return {
        "workload": (f"{wl.name}: one {s.W}x{s.H} RGB uint8 image per GPU per step "
                     f"({wl.n_patches[0]} patches, {wl.n_vis[0]} visual tokens); ViT Q/K bf16 "
                     f"[{wl.n_patches[0]},16,80]; LLM Q bf16 [{s.tq},28,128], K bf16 [{wl.n_vis[0]},4,128]; "
                     f"embeddings bf16 [{wl.n_vis[0]},3584]; keep {keep:.0%}"),
        "images_per_step_per_gpu": 1,
        "keep_fraction": keep,
        "l2": "flushed before every timed step by a 256 MiB device write",
        "timing": "CUDA events on the launching stream around each step; each libpace call replayed from a CUDA graph",
    }


class ClockSampler:
    """nvidia-smi clock / throttle sampling during a timed region."""
    QUERY = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
             "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
             "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, device_index):
        self.dev = device_index
        self.proc = None
        self.path = None

    def start(self):
        fd, self.path = tempfile.mkstemp(suffix=".csv")
        os.close(fd)
        try:
            self.proc = subprocess.Popen(["nvidia-smi", f"--query-gpu={self.QUERY}", "--format=csv,noheader,nounits",
                                          "-i", str(self.dev), "-lms", "100"],
                                         stdout=open(self.path, "w"), stderr=subprocess.DEVNULL)
        except OSError:
            self.proc = None
        time.sleep(0.3)

    def stop(self):
        if self.proc is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"], "samples": 0}
        time.sleep(0.2)
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
        sm, smax, power, reasons = [], [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        with open(self.path) as f:
            for line in f:
                parts = [p.strip() for p in line.split(",")]
                if len(parts) < 9:
                    continue
                try:
                    sm.append(float(parts[1]))
                    smax.append(float(parts[2]))
                    power.append(float(parts[3]))
                except ValueError:
                    continue
                for n, v in zip(names, parts[5:9]):
                    if v.lower() == "active":
                        reasons.add(n)
        os.unlink(self.path)
        return {"sm_mhz": statistics.median(sm) if sm else None, "sm_max_mhz": max(smax) if smax else None,
                "power_w_max": max(power) if power else None, "reasons": sorted(reasons), "samples": len(sm)}


def max_over_ranks(x: float, world: int, device) -> float:
    """Maximum of a per-rank scalar over all ranks (the slowest rank sets the job time)."""
    if world <= 1:
        return float(x)
    import torch
    import torch.distributed as dist
    t = torch.tensor([float(x)], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def per_image_us(total_ms: float, steps: int, world: int, images_per_step: int = 1) -> float:
    """Whole-job time per image: every rank processes images_per_step images per step."""
    return total_ms * 1e3 / (steps * world * images_per_step)


# ----------------------------------------------------------------------------------------------
# CPU oracle sample (the reference arm and the cpu_baseline leg)
# ----------------------------------------------------------------------------------------------
def oracle_sample(wl, keep, vit_rows=2048, crop_div=4):
    """Times the fp64 oracle on a bounded sample of one image and scales it to a whole image.

    density : oracle on a centred crop with 1/crop_div of each side, scaled by (N/N_crop)^2
              (Eq. 1 is a double sum over all token pairs);
    resample: whole image to the oracle's target size;
    S_vis   : one head, the first vit_rows query rows against all keys, scaled by
              heads x N / vit_rows;
    S_llm, fusion, top-K, gather: whole image.
    """
    from oracle import pace_oracle as O
    from paper_2608_27206_gb300 import synth
    img = wl.images[0]
    H, W = img.shape[:2]
    t = {}
    ch, cw = (H // crop_div) // 14 * 14, (W // crop_div) // 14 * 14
    y0, x0 = (H - ch) // 2 // 14 * 14, (W - cw) // 2 // 14 * 14
    crop = np.ascontiguousarray(img[y0:y0 + ch, x0:x0 + cw])
    n_full, n_crop = (H // 14) * (W // 14), (ch // 14) * (cw // 14)
    t0 = time.perf_counter()
    O.apc_density(crop)
    t["density"] = (time.perf_counter() - t0) * (n_full / n_crop) ** 2
    st = O.apc_density_tokens(O.patch_tokens(crop))
    ho, wo = O.target_size(H, W, O.retention_ratio(st["rho"]))
    t0 = time.perf_counter()
    O.apc_resample(img, ho, wo)
    t["resample"] = time.perf_counter() - t0
    q = synth.bf16_bits_to_f64(wl.vit_q[:vit_rows, 0])
    k = synth.bf16_bits_to_f64(wl.vit_k[:, 0])
    t0 = time.perf_counter()
    O.received_attention(q, k, 1 / math.sqrt(80))
    t["vit"] = (time.perf_counter() - t0) * wl.vit_q.shape[1] * (wl.vit_q.shape[0] / vit_rows)
    ql, kl = synth.bf16_bits_to_f64(wl.llm_q), synth.bf16_bits_to_f64(wl.llm_k)
    t0 = time.perf_counter()
    s_llm = O.llm_text_visual_importance(ql, kl, wl.cu_q, wl.cu_vis, 1 / math.sqrt(128))
    t["llm"] = time.perf_counter() - t0
    s_vis = np.random.default_rng(0).lognormal(size=wl.n_vis[0])  # stand-in map for timing only
    K = O.budget(wl.n_vis[0], keep)
    t0 = time.perf_counter()
    sel = O.ddae_select(s_llm, s_vis, wl.cu_vis, [K])
    t["select"] = time.perf_counter() - t0
    t0 = time.perf_counter()
    O.gather_rows(wl.embed, sel["kept"])
    t["gather"] = time.perf_counter() - t0
    total = sum(t.values())
    sample = (f"fp64 numpy oracle on the host cores: density on a {cw}x{ch} centre crop scaled by (N/N_crop)^2, "
              f"resample of the whole image, S_vis for 1 of 16 heads x {vit_rows} of {wl.vit_q.shape[0]} query rows "
              f"scaled linearly, S_llm / fusion / top-K / gather on the whole image")
    return total, t, sample


def run_reference(args):
    rank = int(os.environ.get("RANK", "0"))
    if rank != 0:
        return 0
    from paper_2608_27206_gb300 import synth
    wl = synth.make_workload(WORKLOAD, seed=0, keep=KEEP, parts=("image", "vit", "llm", "embed"))
    for _ in range(args.warmup):
        oracle_sample(wl, KEEP, vit_rows=args.ref_vit_rows)
    times, parts, sample = [], None, ""
    for _ in range(args.steps):
        tot, parts, sample = oracle_sample(wl, KEEP, vit_rows=args.ref_vit_rows)
        times.append(tot)
    per_image_s = float(np.mean(times))
    value = per_image_s * 1e6
    line = {
        "impl": "reference", "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": args.gpus,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": per_image_s * 1e3, "higher_is_better": False,
        "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
        "config": workload_config(wl, KEEP),
        "cpu_baseline": {"value": value, "unit": UNIT, "cores": os.cpu_count(), "kind": "oracle", "sample": sample,
                         "parts_s": {k: round(v, 4) for k, v in parts.items()}},
        "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line))
    return 0


# ----------------------------------------------------------------------------------------------
# GPU arm
# ----------------------------------------------------------------------------------------------
def capture_graphs(pipe):
    """One CUDA graph per libpace call of the step, captured after an eager warm-up."""
    import torch
    s = torch.cuda.Stream()
    s.wait_stream(torch.cuda.current_stream())
    with torch.cuda.stream(s):
        pipe.step()
    torch.cuda.current_stream().wait_stream(s)
    torch.cuda.synchronize()
    graphs = []
    for name, f in pipe.parts:
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g):
            f()
        graphs.append((name, g))
    torch.cuda.synchronize()
    return graphs


def algorithmic_counts(wl, keep, r_ratio):
    """Algorithmic flops / bytes per step (one image), per part."""
    n, nv = wl.n_patches[0], wl.n_vis[0]
    H, W = wl.specs[0].H, wl.specs[0].W
    tq = wl.specs[0].tq
    K = int(math.floor(keep * nv + 0.5))
    img_bytes = H * W * 3
    s = math.sqrt(max(r_ratio, 0.0))
    ho = min(H, max(28, 28 * int(math.floor(H * s / 28 + 0.5))))
    wo = min(W, max(28, 28 * int(math.floor(W * s / 28 + 0.5))))
    return {
        "vit_flops": 2 * 2 * n * n * 80 * 16,            # two passes of 2 N^2 d H
        "vit_ex2": 2 * n * n * 16,                          # one exp2 per score and pass
        "llm_flops": 2 * 2 * tq * 28 * nv * 128,
        "density_bytes": img_bytes + 4 * n,                # image once + d_i
        "resample_bytes": img_bytes + ho * wo * 3,
        "select_bytes": 2 * 4 * nv + 4 * nv + 4 * K,       # two raw maps in, S_final + kept out
        "gather_bytes": 2 * K * 3584 * 2,
    }


def measure_next_rows(P, device, flush, peak_tf, hbm_gbs, reps=10):
    """Times the calls of the paths beyond the step (preview-token density, full-sequence S_llm,
    the prune step's gathers) on the 4K image's shapes, each replayed from a CUDA graph with L2
    flushed before every replay; median over `reps`.  Inputs are seeded device tensors."""
    import torch
    from paper_2608_27206_gb300 import synth
    g = torch.Generator(device=device)
    g.manual_seed(1234)

    def randn(*shape, scale=1.0):
        return (torch.randn(*shape, generator=g, device=device) * scale).to(torch.bfloat16)

    def timed(fn):
        fn()
        torch.cuda.synchronize()
        st = torch.cuda.Stream(device)
        with torch.cuda.stream(st):
            gr = torch.cuda.CUDAGraph()
            with torch.cuda.graph(gr, stream=st):
                fn()
        torch.cuda.synchronize()
        ts = []
        for _ in range(reps):
            flush.zero_()
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e0.record()
            gr.replay()
            e1.record()
            torch.cuda.synchronize()
            ts.append(e0.elapsed_time(e1))
        return statistics.median(ts) * 1e-3   # seconds

    out = {}
    # f1: APC density on preview tokens: 42196 tokens x 1280 (ViT hidden width), bf16
    n_tok, dim = 42196, 1280
    T = randn(n_tok, dim)
    cu = [0, n_tok]
    d = torch.empty(n_tok, dtype=torch.float32, device=device)
    st = torch.zeros((1, 10), dtype=torch.int32, device=device)
    ws = torch.empty(max(P.pace_apc_density_tokens_workspace_size(cu, dim), 16), dtype=torch.uint8, device=device)
    sec = timed(lambda: P.pace_apc_density_tokens(T, cu, [3836], [2156], d_out=d, stats=st, ws=ws))
    nbytes = 2 * n_tok * dim * 2 + 4 * n_tok
    out["f1_density_tokens"] = {"shape": f"T bf16 [{n_tok},{dim}]", "us": round(sec * 1e6, 2), "bound": "hbm",
                                "bytes": nbytes, "achieved": round(nbytes / sec / 1e9, 1), "unit": "GB/s",
                                "frac": round(nbytes / sec / 1e9 / hbm_gbs, 4)}
    del T, ws
    # f1: APC density with the four pixel-statistic previews on the 4K image (HBM roofline: the
    # image read once + 32 B of token written and read twice per patch + d)
    img = torch.randint(0, 256, (2156 * 3836 * 3,), generator=g, device=device, dtype=torch.uint8)
    wsp = torch.empty(max(P.pace_apc_density_pixel_workspace_size([2156], [3836]), 16), dtype=torch.uint8,
                      device=device)
    for feat in P.PIXEL_FEATURES:
        sec = timed(lambda: P.pace_apc_density_pixel(img, [0], [2156], [3836], feat, d_out=d, stats=st, ws=wsp))
        nbytes = img.numel() + n_tok * (3 * 32 + 4)
        out[f"f1_density_pixel_{feat}"] = {"shape": "3836x2156 RGB uint8", "us": round(sec * 1e6, 2),
                                           "bound": "hbm", "bytes": nbytes,
                                           "achieved": round(nbytes / sec / 1e9, 1), "unit": "GB/s",
                                           "frac": round(nbytes / sec / 1e9 / hbm_gbs, 4)}
    del img, wsp, d
    # f2: full-sequence S_llm (Vision+Text queries, causal): system 20 + 10549 visual + 256 text
    v, nv, nt = 20, 10549, 256
    S = v + nv + nt
    Q = randn(S, 28, 128)
    K = randn(S, 4, 128)
    o = torch.empty(nv, dtype=torch.float32, device=device)
    wsq = torch.empty(max(P.pace_llm_sequence_importance_workspace_size([0, S], [v], [nv], 28, 4), 16),
                      dtype=torch.uint8, device=device)
    sec = timed(lambda: P.pace_llm_sequence_importance(Q, K, [0, S], [v], [nv], "vision_text", out=o, ws=wsq))
    # pass 1: query at position p (p >= v) sees p + 1 keys; pass 2: visual key at position q is
    # seen by the S - q queries at or after it
    pairs1 = sum(p + 1 for p in range(v, S))
    pairs2 = sum(S - q for q in range(v, v + nv))
    flops = 2 * 128 * 28 * (pairs1 + pairs2)
    out["f2_sequence_importance"] = {"shape": f"Q bf16 [{S},28,128], K bf16 [{S},4,128], vision_text",
                                     "us": round(sec * 1e6, 2), "bound": "tensor", "flops": flops,
                                     "achieved": round(flops / sec / 1e12, 1), "unit": "TFLOP/s",
                                     "frac": round(flops / sec / 1e12 / peak_tf, 4)}
    del Q, K, o, wsq
    # f3: prune step: row list + one gather of hidden states [S, 3584], the K and V rows of layers
    # 0..2 ([S, 4, 128] each) and the M-RoPE ids [3, S] (int64), keep 10 % of the visual tokens
    keep = P.pace_budget(nv, 0.10)
    kept = torch.sort(torch.randperm(nv, generator=g, device=device)[:keep])[0].to(torch.int32)
    n_out = S - nv + keep
    idx = torch.empty(n_out, dtype=torch.int32, device=device)
    hid = randn(S, 3584)
    kv = [randn(S, 4, 128) for _ in range(6)]
    pos = torch.arange(3 * S, device=device, dtype=torch.int64).view(3, S)
    hid_o = torch.empty(n_out, 3584, dtype=torch.bfloat16, device=device)
    kv_o = [torch.empty(n_out, 4, 128, dtype=torch.bfloat16, device=device) for _ in range(6)]
    pos_o = torch.empty(3, n_out, dtype=torch.int64, device=device)
    specs = [P.gather_spec(hid, hid_o, 0)] + [P.gather_spec(a, b, 0) for a, b in zip(kv, kv_o)] + \
            [P.gather_spec(pos, pos_o, 1)]

    def prune():
        P.pace_prune_index([0, S], [v], [0, nv], [0, keep], kept, out=idx)
        P.pace_gather_multi(specs, idx)
    sec = timed(prune)
    nbytes = 2 * n_out * (3584 * 2 + 6 * 4 * 128 * 2 + 3 * 8) + 4 * keep + 4 * n_out
    out["f3_prune_gather"] = {"shape": f"{n_out} of {S} rows: hidden [S,3584] + 6 KV [S,4,128] bf16 + ids [3,S]",
                              "us": round(sec * 1e6, 2), "bound": "hbm", "bytes": nbytes,
                              "achieved": round(nbytes / sec / 1e9, 1), "unit": "GB/s",
                              "frac": round(nbytes / sec / 1e9 / hbm_gbs, 4)}
    del hid, kv, hid_o, kv_o, pos, pos_o
    # a5/a6 on batches (one 4K map is latency-bound at 131 KB): the 16-image ragged batch's map
    # sizes and keep fractions, and 64 copies of the 4K image's map; positive random scores
    for name, nvs, fracs in (("a5a6_select_ragged16", [s.H // synth.MERGE_PX * (s.W // synth.MERGE_PX)
                                                      for s in synth.workload_specs("ragged16")],
                              [s.keep for s in synth.workload_specs("ragged16")]),
                             ("a5a6_select_img4k_x64", [nv] * 64, [0.10] * 64)):
        cu_v = np.concatenate([[0], np.cumsum(nvs)]).astype(np.int32)
        ks = [P.pace_budget(n, f) for n, f in zip(nvs, fracs)]
        cu_k = np.concatenate([[0], np.cumsum(ks)]).astype(np.int32)
        tot = int(cu_v[-1])
        s_llm = torch.rand(tot, generator=g, device=device) * 8
        s_vis = torch.rand(tot, generator=g, device=device).pow(3) * 16
        sf = torch.empty(tot, dtype=torch.float32, device=device)
        wts = torch.empty((len(nvs), 2), dtype=torch.float32, device=device)
        kp = torch.empty(int(cu_k[-1]), dtype=torch.int32, device=device)
        sec = timed(lambda: P.pace_ddae_select(s_llm, s_vis, cu_v, cu_k, s_final=sf, weights=wts, kept=kp))
        nbytes = 3 * 4 * tot + 4 * int(cu_k[-1]) + 8 * len(nvs)
        out[name] = {"shape": f"{len(nvs)} maps, {tot} scores, keep {int(cu_k[-1])}", "us": round(sec * 1e6, 2),
                     "bound": "hbm", "bytes": nbytes, "achieved": round(nbytes / sec / 1e9, 1), "unit": "GB/s",
                     "frac": round(nbytes / sec / 1e9 / hbm_gbs, 4)}
    return out


def run_gpu(args):
    import torch
    import torch.distributed as dist
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    if world > 1:
        torch.cuda.set_device(local)
        dist.init_process_group("nccl", device_id=torch.device("cuda", local))
    else:
        torch.cuda.set_device(0)
    device = torch.device("cuda", torch.cuda.current_device())
    from paper_2608_27206_gb300 import build as pace_build
    pace_build.build()
    from paper_2608_27206_gb300 import pace as P
    from paper_2608_27206_gb300 import synth
    P.pace_init(torch.cuda.current_device())

    from paper_2608_27206_gb300.hotpath import HotPath
    wl = synth.make_workload(WORKLOAD, seed=rank, keep=KEEP)
    pipe = HotPath(wl, device)
    flush = torch.empty(FLUSH_BYTES, dtype=torch.uint8, device=device)

    # launches per step (eager), then graphs
    c0 = P.pace_kernel_launch_count()
    pipe.step()
    torch.cuda.synchronize()
    launches_per_step = P.pace_kernel_launch_count() - c0
    graphs = capture_graphs(pipe)
    for _ in range(args.warmup):
        flush.zero_()
        for _, g in graphs:
            g.replay()
    torch.cuda.synchronize()
    code, where = P.pace_device_status(clear=True)
    if code != 0:
        raise RuntimeError(f"device status {code} from kernel {where} during warm-up")

    nparts = len(graphs)
    ev = [[torch.cuda.Event(enable_timing=True) for _ in range(nparts + 1)] for _ in range(args.steps)]
    sampler = ClockSampler(torch.cuda.current_device())
    sampler.start()
    if world > 1:
        dist.barrier()
    torch.cuda.synchronize()
    t_wall0 = time.perf_counter()
    for k in range(args.steps):
        flush.zero_()
        ev[k][0].record()
        for i, (_, g) in enumerate(graphs):
            g.replay()
            ev[k][i + 1].record()
    torch.cuda.synchronize()
    if world > 1:
        dist.barrier()
    t_wall = time.perf_counter() - t_wall0
    clocks = sampler.stop()
    part_ms = {name: [] for name, _ in graphs}
    step_ms = []
    for k in range(args.steps):
        step_ms.append(ev[k][0].elapsed_time(ev[k][nparts]))
        for i, (name, _) in enumerate(graphs):
            part_ms[name].append(ev[k][i].elapsed_time(ev[k][i + 1]))
    total_ms = max_over_ranks(float(sum(step_ms)), world, device)
    ms_per_step = total_ms / args.steps
    value = per_image_us(total_ms, args.steps, world)

    # correctness guard on the timed outputs
    code, where = P.pace_device_status(clear=True)
    if code != 0:
        raise RuntimeError(f"device status {code} from kernel {where} in the timed region")
    stats = P.stats_dict(pipe.stats)[0]

    # e2e: pinned host inputs -> device, the public calls, results -> pinned host
    pinned = {k: v.pin_memory() for k, v in pipe.host.items()}
    out_host = {"kept": torch.empty(tuple(pipe.kept.shape), dtype=torch.int32).pin_memory(),
                "rows": torch.empty(tuple(pipe.rows.shape), dtype=torch.bfloat16).pin_memory(),
                "stats": torch.empty((1, 10), dtype=torch.int32).pin_memory(),
                "s_final": torch.empty(pipe.s_final.numel(), dtype=torch.float32).pin_memory()}
    h2d = sum(v.numel() * v.element_size() for v in pinned.values())
    d2h = sum(v.numel() * v.element_size() for v in out_host.values())

    copy_stream, readback_stream = torch.cuda.Stream(device), torch.cuda.Stream(device)

    def e2e_step():
        # returns the event after which the step's results are in the pinned host tensors
        return pipe.step_from_host(pinned, out_host, copy_stream, readback_stream)

    for _ in range(max(1, args.warmup)):
        e2e_step()
    torch.cuda.synchronize()
    e_start, e_end = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    if world > 1:
        dist.barrier()
    torch.cuda.synchronize()
    e_start.record()
    copy_stream.wait_event(e_start)       # no copy of the timed steps starts before the clock
    for _ in range(args.steps):
        last = e2e_step()
    torch.cuda.current_stream(device).wait_event(last)     # every step's results are on the host
    e_end.record()
    torch.cuda.synchronize()
    e2e_ms = max_over_ranks(e_start.elapsed_time(e_end), world, device)
    if world > 1:
        dist.barrier()
    e2e_value = per_image_us(e2e_ms, args.steps, world)
    # single-image latency: one step from host memory with nothing else in flight
    lat = []
    for _ in range(3):
        torch.cuda.synchronize()
        l0, l1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        l0.record()
        torch.cuda.current_stream(device).wait_event(e2e_step())
        l1.record()
        torch.cuda.synchronize()
        lat.append(l0.elapsed_time(l1))
    latency_us = max_over_ranks(statistics.median(lat), world, device) * 1e3

    if rank == 0:
        peaks, peak_src = load_peaks()
        cnt = algorithmic_counts(wl, KEEP, stats["r"])
        vit_ms = statistics.mean(part_ms["vit"])
        achieved = cnt["vit_flops"] / (vit_ms * 1e-3) / 1e12
        # MUFU ceiling: 32 ex2 per clock per SM (measured on GB300) at the median SM clock seen
        sm_mhz = (clocks or {}).get("sm_mhz") or float(peaks.get("sm_max_mhz", 0) or 0)
        mufu_peak = 32.0 * torch.cuda.get_device_properties(0).multi_processor_count * sm_mhz * 1e6 if sm_mhz else None
        peak = float(peaks.get("bf16_tflops", FALLBACK_PEAKS["bf16_tflops"]))
        hbm = float(peaks.get("hbm_gbs", FALLBACK_PEAKS["hbm_gbs"]))
        mean = {k: statistics.mean(v) for k, v in part_ms.items()}
        other = {}
        for name, key in (("density", "density_bytes"), ("resample", "resample_bytes"), ("select", "select_bytes"),
                          ("gather", "gather_bytes")):
            gbs = cnt[key] / (mean[name] * 1e-3) / 1e9
            other[name] = {"bound": "hbm", "us": round(mean[name] * 1e3, 2), "achieved": round(gbs, 1),
                           "peak": hbm, "unit": "GB/s", "frac": round(gbs / hbm, 4), "bytes": cnt[key]}
        llm_tf = cnt["llm_flops"] / (mean["llm"] * 1e-3) / 1e12
        other["llm"] = {"bound": "tensor", "us": round(mean["llm"] * 1e3, 2), "achieved": round(llm_tf, 1),
                        "peak": peak, "unit": "TFLOP/s", "frac": round(llm_tf / peak, 4), "flops": cnt["llm_flops"]}
        nxt = measure_next_rows(P, device, flush, peak, hbm) if world == 1 and not args.no_next_rows else None
        cpu = None
        if world == 1 and not args.no_cpu_baseline:
            tot, parts, sample = oracle_sample(wl, KEEP, vit_rows=args.ref_vit_rows)
            cpu = {"value": tot * 1e6, "unit": UNIT, "cores": os.cpu_count(), "kind": "oracle", "sample": sample,
                   "parts_s": {k: round(v, 4) for k, v in parts.items()}}
        line = {
            "metric": METRIC, "value": round(value, 3), "unit": UNIT, "n_gpus": world, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": round(ms_per_step, 4), "higher_is_better": False,
            "scaling": "weak", "vs_baseline": None, "dtype": "bf16", "data": "synthetic",
            "config": workload_config(wl, KEEP),
            "roofline": {"bound": "tensor", "achieved": round(achieved, 1), "peak": peak, "unit": "TFLOP/s",
                         "frac": round(achieved / peak, 4), "traffic": profiled_traffic(),
                         "traffic_unit": "bytes per call (ncu dram read+write, profiles/vit_importance_img4k.md)",
                         "kernel": "ViT received attention (attn_row_lse + attn_colsum + attn_reduce), one launch "
                                   "of pace_vit_attn_importance",
                         "algorithmic_flops": cnt["vit_flops"], "us": round(vit_ms * 1e3, 1),
                         # one pass of QK^T is the "useful" work; the second pass recomputes it
                         "useful_one_pass_frac": round(achieved / 2 / peak, 4),
                         # every score costs one exp2 per pass (N^2 H per pass)
                         "mufu_ex2_per_s": round(cnt["vit_ex2"] / (vit_ms * 1e-3), 1),
                         "mufu_frac": round(cnt["vit_ex2"] / (vit_ms * 1e-3) / mufu_peak, 4)
                         if mufu_peak else None,
                         "mufu_peak_ex2_per_s": mufu_peak,
                         "peak_source": f"{peak_src} bf16 dense burst (MEASURED_PEAKS.json)"
                         if peak_src == "measured" else "fallback 1.9 PFLOP/s bf16"},
            "rooflines_other": other,
            "next_rows": nxt,
            "breakdown_us": {k: round(v * 1e3, 2) for k, v in mean.items()},
            "visual_tokens_scored_per_s": round(wl.n_vis[0] * world / (ms_per_step * 1e-3), 1),
            "cpu_baseline": cpu,
            "e2e": {"value": round(e2e_value, 3), "unit": UNIT, "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h,
                    "pipelining": "two device input slots: image n+1's host-to-device copies run during image "
                                  "n's calls; every step's copies and result read-back are inside the timed region",
                    "latency_us_one_image": round(latency_us, 1)},
            "gpu_launches": launches_per_step * args.steps,
            "clocks": clocks,
            "apc": {"rho": round(stats["rho"], 5), "r": round(stats["r"], 5),
                    "target": [stats["h_out"], stats["w_out"]]},
            "wall_s_timed_region": round(t_wall, 4),
        }
        print(json.dumps(line))
    if world > 1:
        dist.destroy_process_group()
    return 0


def run_profile(args):
    """Runs one libpace call `--reps` times on the workload (for ncu captures; prints no result)."""
    import torch
    torch.cuda.set_device(0)
    from paper_2608_27206_gb300 import build as pace_build
    pace_build.build()
    from paper_2608_27206_gb300 import pace as P
    from paper_2608_27206_gb300 import synth
    P.pace_init(0)
    wl = synth.make_workload(args.workload, seed=0, keep=KEEP)
    from paper_2608_27206_gb300.hotpath import HotPath
    pipe = HotPath(wl, torch.device("cuda", 0))
    fns = dict(pipe.parts)
    needs = {"resample": ["density"], "select": ["vit", "llm"], "gather": ["vit", "llm", "select"]}
    for name in needs.get(args.profile, []):      # producers of this call's inputs
        fns[name]()
    for _ in range(args.reps):
        fns[args.profile]()
    torch.cuda.synchronize()
    code, where = P.pace_device_status(clear=True)
    if code != 0:
        raise RuntimeError(f"device status {code} from kernel {where}")
    return 0


def main():
    ap = argparse.ArgumentParser(description=__doc__.split("\n")[0])
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=200)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", choices=("ours", "reference"), default="ours")
    ap.add_argument("--ref-vit-rows", type=int, default=2048)
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-next-rows", action="store_true", help="skip the timing of the NEXT-row calls")
    ap.add_argument("--profile", choices=("density", "resample", "vit", "llm", "select", "gather"),
                    help="run only this call --reps times (for profiler captures)")
    ap.add_argument("--reps", type=int, default=1)
    ap.add_argument("--workload", default=WORKLOAD)
    args = ap.parse_args()
    if args.profile:
        return run_profile(args)
    if args.warmup < 3:
        ap.error("--warmup must be at least 3")
    if args.impl == "reference":
        return run_reference(args)
    return run_gpu(args)


if __name__ == "__main__":
    sys.exit(main())
