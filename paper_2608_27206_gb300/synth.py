"""Seeded synthetic inputs shaped like Qwen2.5-VL-7B workloads.

This module only draws inputs.  It holds none of the method's arithmetic: the
CUDA path and the fp64 oracle both receive exactly the arrays built here.

Workloads (the five shapes the hot path is measured and checked on):

  img448      448x448 image, 4x4 tiles, 50 % high-frequency; ViT Q/K [1024,16,80];
              LLM Q [64,28,128], K [256,4,128]; keep 10 %.
  img1344     1344x1344, 8x8 tiles, 30 % HF; ViT [9216,16,80]; LLM Tq=128,
              K [2304,4,128]; keep 25 %.
  frame1904   1904x1064 frame, 16x9 tiles, 20 % HF plus 8 saturated "sink"
              patches whose ViT K rows (and the LLM K rows of the merged tokens
              holding them) carry 4x norm; LLM Tq=96; keep 10 %.
  img4k       3836x2156, 32x18 tiles, 15 % HF; ViT [42196,16,80]; LLM Tq=256,
              K [10549,4,128]; keep 5 % and 10 %.
  ragged16    16 images, H and W drawn as multiples of 28 in [448, 2240],
              10-60 % HF, Tq in [32, 256], keep drawn from {5, 10, 25} %.

Recipe (identical for every workload):
  * image tiles: tile edges at floor(k*W/tx), floor(k*H/ty); exactly
    round(frac * tiles) tiles, picked at random, are i.i.d. uniform uint8
    noise; the others are a linear RGB gradient between two uniform random
    endpoints along a uniform random direction, rounded to uint8.
  * Q and K entries are i.i.d. N(0,1) in fp32; every token row (all heads) is
    multiplied by one LogNormal(0, 0.5) factor; values are rounded to bf16
    (round-to-nearest-even).  Embedding rows E are bf16 N(0,1).
  * ViT rows are in merge-grouped order: the 4 patches of one 2x2 merge unit
    are consecutive, merge units in raster order.
Every array is drawn from numpy's PCG64 seeded by (seed, workload, part).
"""
from __future__ import annotations

from dataclasses import dataclass, field
from typing import List, Optional

import numpy as np

PATCH = 14
MERGE_PX = 28
VIT_HEADS, VIT_DIM = 16, 80
LLM_QHEADS, LLM_KVHEADS, LLM_DIM = 28, 4, 128
EMBED_DIM = 3584

WORKLOADS = ("img448", "img1344", "frame1904", "img4k", "ragged16")
_WID = {n: i for i, n in enumerate(WORKLOADS)}
_PART = {"image": 1, "vit": 2, "llm": 3, "embed": 4, "meta": 5, "sink": 6}


def _rng(seed: int, workload: str, part: str, index: int = 0) -> np.random.Generator:
    return np.random.Generator(np.random.PCG64([seed, _WID.get(workload, 99), _PART[part], index]))


# ----------------------------------------------------------------------------------------------
# bf16 storage helpers (format conversion only)
# ----------------------------------------------------------------------------------------------
def f32_to_bf16_bits(x: np.ndarray) -> np.ndarray:
    """Round fp32 values to bf16, round-to-nearest-even; returns uint16 bit patterns."""
    u = np.ascontiguousarray(x, dtype=np.float32).view(np.uint32).reshape(-1)
    out = np.empty(u.shape, dtype=np.uint16)
    step = 1 << 20                       # cache-sized chunks
    for i in range(0, u.size, step):
        c = u[i:i + step]
        r = (c >> 16) & np.uint32(1)
        r += np.uint32(0x7FFF)
        r += c                           # finite inputs never wrap: 0xFF7FFFFF + 0x8000 < 2**32
        r >>= 16
        out[i:i + step] = r
    return out.reshape(np.shape(x))


def bf16_bits_to_f64(b: np.ndarray) -> np.ndarray:
    """Exact widening of bf16 bit patterns to float64."""
    return (b.astype(np.uint32) << 16).view(np.float32).astype(np.float64)


# ----------------------------------------------------------------------------------------------
# Images
# ----------------------------------------------------------------------------------------------
def make_image(rng: np.random.Generator, H: int, W: int, tx: int, ty: int, hf_frac: float) -> np.ndarray:
    """Tile image: round(hf_frac*tx*ty) noise tiles, gradient tiles elsewhere.  uint8 [H, W, 3]."""
    img = np.empty((H, W, 3), dtype=np.uint8)
    n_tiles = tx * ty
    n_hf = int(np.floor(hf_frac * n_tiles + 0.5))
    hf = np.zeros(n_tiles, dtype=bool)
    hf[rng.permutation(n_tiles)[:n_hf]] = True
    xs = [(k * W) // tx for k in range(tx + 1)]
    ys = [(k * H) // ty for k in range(ty + 1)]
    for j in range(ty):
        for i in range(tx):
            y0, y1, x0, x1 = ys[j], ys[j + 1], xs[i], xs[i + 1]
            h, w = y1 - y0, x1 - x0
            if h == 0 or w == 0:
                continue
            if hf[j * tx + i]:
                img[y0:y1, x0:x1] = rng.integers(0, 256, size=(h, w, 3), dtype=np.uint8)
            else:
                c0 = rng.uniform(0, 255, size=3)
                c1 = rng.uniform(0, 255, size=3)
                th = rng.uniform(0, 2 * np.pi)
                yy, xx = np.mgrid[0:h, 0:w].astype(np.float64)
                proj = xx * np.cos(th) + yy * np.sin(th)
                lo, hi = proj.min(), proj.max()
                t = (proj - lo) / (hi - lo) if hi > lo else np.zeros_like(proj)
                val = c0[None, None, :] + t[:, :, None] * (c1 - c0)[None, None, :]
                img[y0:y1, x0:x1] = np.clip(np.rint(val), 0, 255).astype(np.uint8)
    return img


def merge_grouped_row(py: int, px: int, gw: int) -> int:
    """Row of patch (py, px) when the 4 patches of a 2x2 merge unit are consecutive."""
    return 4 * ((py // 2) * (gw // 2) + px // 2) + 2 * (py % 2) + (px % 2)


# ----------------------------------------------------------------------------------------------
# Q / K / E
# ----------------------------------------------------------------------------------------------
def make_qk(rng: np.random.Generator, rows: int, heads: int, dim: int,
            boost_rows: Optional[np.ndarray] = None, boost: float = 4.0) -> np.ndarray:
    """bf16 bits [rows, heads, dim]: N(0,1) entries times a LogNormal(0,0.5) per-row factor."""
    x = rng.standard_normal(size=(rows, heads, dim), dtype=np.float32)
    s = rng.lognormal(0.0, 0.5, size=rows).astype(np.float32)
    if boost_rows is not None and len(boost_rows):
        s[boost_rows] *= np.float32(boost)
    step = max(1, (1 << 20) // max(1, heads * dim))
    for i in range(0, rows, step):
        x[i:i + step] *= s[i:i + step, None, None]
    return f32_to_bf16_bits(x)


def make_embed(rng: np.random.Generator, rows: int, dim: int = EMBED_DIM) -> np.ndarray:
    return f32_to_bf16_bits(rng.standard_normal(size=(rows, dim), dtype=np.float32))


# ----------------------------------------------------------------------------------------------
# Workloads
# ----------------------------------------------------------------------------------------------
@dataclass
class ImageSpec:
    H: int
    W: int
    tx: int
    ty: int
    hf: float
    tq: int
    keep: float
    sinks: int = 0


@dataclass
class Workload:
    name: str
    seed: int
    specs: List[ImageSpec]
    images: List[np.ndarray] = field(default_factory=list)
    sink_patches: List[np.ndarray] = field(default_factory=list)   # per image: [n, 2] (py, px)
    vit_q: Optional[np.ndarray] = None      # bf16 bits [sum N, 16, 80]
    vit_k: Optional[np.ndarray] = None
    llm_q: Optional[np.ndarray] = None      # bf16 bits [sum Tq, 28, 128]
    llm_k: Optional[np.ndarray] = None      # bf16 bits [sum Nv, 4, 128]
    embed: Optional[np.ndarray] = None      # bf16 bits [sum Nv, 3584]

    @property
    def B(self) -> int:
        return len(self.specs)

    @property
    def n_patches(self) -> List[int]:
        return [(s.H // PATCH) * (s.W // PATCH) for s in self.specs]

    @property
    def n_vis(self) -> List[int]:
        return [(s.H // MERGE_PX) * (s.W // MERGE_PX) for s in self.specs]

    @property
    def cu_patches(self) -> np.ndarray:
        return np.concatenate([[0], np.cumsum(self.n_patches)]).astype(np.int32)

    @property
    def cu_vis(self) -> np.ndarray:
        return np.concatenate([[0], np.cumsum(self.n_vis)]).astype(np.int32)

    @property
    def cu_q(self) -> np.ndarray:
        return np.concatenate([[0], np.cumsum([s.tq for s in self.specs])]).astype(np.int32)

    @property
    def keep_fracs(self) -> List[float]:
        return [s.keep for s in self.specs]


def workload_specs(name: str, seed: int = 0, keep: Optional[float] = None) -> List[ImageSpec]:
    if name == "img448":
        specs = [ImageSpec(448, 448, 4, 4, 0.50, 64, 0.10)]
    elif name == "img1344":
        specs = [ImageSpec(1344, 1344, 8, 8, 0.30, 128, 0.25)]
    elif name == "frame1904":
        specs = [ImageSpec(1064, 1904, 16, 9, 0.20, 96, 0.10, sinks=8)]
    elif name == "img4k":
        specs = [ImageSpec(2156, 3836, 32, 18, 0.15, 256, 0.10)]
    elif name == "ragged16":
        r = _rng(seed, name, "meta")
        specs = []
        for _ in range(16):
            H = MERGE_PX * int(r.integers(16, 81))
            W = MERGE_PX * int(r.integers(16, 81))
            hf = float(r.uniform(0.10, 0.60))
            tq = int(r.integers(32, 257))
            kp = float(r.choice([0.05, 0.10, 0.25]))
            specs.append(ImageSpec(H, W, max(2, round(W / 224)), max(2, round(H / 224)), hf, tq, kp))
    else:
        raise ValueError(f"unknown workload {name!r}")
    if keep is not None:
        for s in specs:
            s.keep = keep
    return specs


def make_workload(name: str, seed: int = 0, parts=("image", "vit", "llm", "embed"),
                  keep: Optional[float] = None) -> Workload:
    """Build the seeded inputs of one workload.  `parts` limits what is drawn."""
    wl = Workload(name, seed, workload_specs(name, seed, keep))
    vit_boost, llm_boost = [], []
    row0, tok0 = 0, 0
    for b, s in enumerate(wl.specs):
        gh, gw = s.H // PATCH, s.W // PATCH
        sinks = np.zeros((0, 2), dtype=np.int64)
        if s.sinks:
            r = _rng(seed, name, "sink", b)
            flat = r.permutation(gh * gw)[: s.sinks]
            sinks = np.stack([flat // gw, flat % gw], axis=1)
            for py, px in sinks:
                vit_boost.append(row0 + merge_grouped_row(int(py), int(px), gw))
                llm_boost.append(tok0 + (int(py) // 2) * (gw // 2) + int(px) // 2)
        wl.sink_patches.append(sinks)
        if "image" in parts:
            img = make_image(_rng(seed, name, "image", b), s.H, s.W, s.tx, s.ty, s.hf)
            for py, px in sinks:
                img[py * PATCH:(py + 1) * PATCH, px * PATCH:(px + 1) * PATCH] = 255
            wl.images.append(img)
        row0 += gh * gw
        tok0 += (gh // 2) * (gw // 2)
    llm_boost = np.unique(np.asarray(llm_boost, dtype=np.int64))
    if "vit" in parts:
        r = _rng(seed, name, "vit")
        n = int(sum(wl.n_patches))
        wl.vit_q = make_qk(r, n, VIT_HEADS, VIT_DIM)
        wl.vit_k = make_qk(r, n, VIT_HEADS, VIT_DIM, np.asarray(vit_boost, dtype=np.int64))
    if "llm" in parts:
        r = _rng(seed, name, "llm")
        wl.llm_q = make_qk(r, int(wl.cu_q[-1]), LLM_QHEADS, LLM_DIM)
        wl.llm_k = make_qk(r, int(wl.cu_vis[-1]), LLM_KVHEADS, LLM_DIM, llm_boost)
    if "embed" in parts:
        wl.embed = make_embed(_rng(seed, name, "embed"), int(wl.cu_vis[-1]))
    return wl


def pack_images(images: List[np.ndarray], align: int = 256):
    """Concatenate HWC uint8 images into one buffer; returns (buffer, byte offsets int64 [B])."""
    offs, pos = [], 0
    for im in images:
        offs.append(pos)
        pos += (im.nbytes + align - 1) // align * align
    buf = np.zeros(max(pos, align), dtype=np.uint8)
    for o, im in zip(offs, images):
        buf[o:o + im.nbytes] = im.reshape(-1)
    return buf, np.asarray(offs, dtype=np.int64)


def random_small_qk(seed: int, rows: int, heads: int, dim: int) -> np.ndarray:
    """bf16 bits for small parity cases of arbitrary shape (same distribution)."""
    return make_qk(np.random.Generator(np.random.PCG64([seed, 7777, rows, heads, dim])), rows, heads, dim)
