"""One step of the condense-and-extract hot path over a batch of images, on the device.

HotPath owns the device copies of a workload's inputs, the outputs and the scratch
buffers, and issues the six libpace calls in pipeline order:

    density -> resample (target size read on the device) -> ViT importance ->
    LLM importance -> DDAE fusion + top-K -> gather of the kept embedding rows

Everything is allocated once in the constructor, so a step only launches kernels and
can be captured in a CUDA graph.  Used by bench.py and by the full-size parity tests,
so both exercise exactly the same calls.
"""
from __future__ import annotations

import math
from typing import Optional, Sequence

import numpy as np
import torch

from . import pace as P
from . import synth


def _bf16(bits: np.ndarray) -> torch.Tensor:
    return torch.from_numpy(np.ascontiguousarray(bits).view(np.int16)).view(torch.bfloat16)


class HotPath:
    def __init__(self, wl: "synth.Workload", device, keep: Optional[Sequence[float]] = None):
        self.wl = wl
        self.dev = torch.device(device)
        self.B = wl.B
        self.H = [im.shape[0] for im in wl.images]
        self.W = [im.shape[1] for im in wl.images]
        buf, off = synth.pack_images(wl.images)
        self.img_off = off
        self.host = {
            "img": torch.from_numpy(buf),
            "vit_q": _bf16(wl.vit_q), "vit_k": _bf16(wl.vit_k),
            "llm_q": _bf16(wl.llm_q), "llm_k": _bf16(wl.llm_k),
            "embed": _bf16(wl.embed),
        }
        self.d = {k: v.to(self.dev) for k, v in self.host.items()}
        self.cu_patches, self.cu_q, self.cu_vis = wl.cu_patches, wl.cu_q, wl.cu_vis
        fracs = list(keep) if keep is not None else wl.keep_fracs
        self.K = [P.pace_budget(n, f) for n, f in zip(wl.n_vis, fracs)]
        self.cu_keep = np.concatenate([[0], np.cumsum(self.K)]).astype(np.int32)
        sizes = [h * w * 3 for h, w in zip(self.H, self.W)]
        self.dst_off = np.concatenate([[0], np.cumsum([(s + 255) // 256 * 256 for s in sizes])])[:-1].astype(np.int64)
        f32, i32, u8 = torch.float32, torch.int32, torch.uint8
        n, nv = int(self.cu_patches[-1]), int(self.cu_vis[-1])
        dev = self.dev
        self.dist = torch.empty(max(n, 1), dtype=f32, device=dev)
        self.stats = torch.zeros((max(self.B, 1), 10), dtype=i32, device=dev)
        self.resized = torch.zeros(int(self.dst_off[-1] + sizes[-1]) if self.B else 1, dtype=u8, device=dev)
        self.s_vis = torch.empty(max(nv, 1), dtype=f32, device=dev)
        self.s_llm = torch.empty(max(nv, 1), dtype=f32, device=dev)
        self.s_final = torch.empty(max(nv, 1), dtype=f32, device=dev)
        self.weights = torch.empty((max(self.B, 1), 2), dtype=f32, device=dev)
        k_tot = int(self.cu_keep[-1])
        self.kept = torch.empty(max(k_tot, 1), dtype=i32, device=dev)
        self.rows = torch.empty((max(k_tot, 1), self.d["embed"].shape[1]), dtype=torch.bfloat16, device=dev)
        self.ws_density = torch.empty(max(P.pace_apc_density_workspace_size(self.H, self.W), 16), dtype=u8,
                                      device=dev)
        self.ws_vit = torch.empty(max(P.pace_vit_attn_importance_workspace_size(self.cu_patches, synth.VIT_HEADS),
                                      16), dtype=u8, device=dev)
        self.ws_llm = torch.empty(max(P.pace_llm_text_visual_importance_workspace_size(
            self.cu_q, self.cu_vis, synth.LLM_QHEADS, synth.LLM_KVHEADS), 16), dtype=u8, device=dev)
        self.parts = [("density", self.density), ("resample", self.resample), ("vit", self.vit),
                      ("llm", self.llm), ("select", self.select), ("gather", self.gather)]

    # -- the six calls ---------------------------------------------------------------------------
    def density(self):
        P.pace_apc_density(self.d["img"], self.img_off, self.H, self.W, d_out=self.dist, stats=self.stats,
                           ws=self.ws_density)

    def resample(self):
        P.pace_apc_resample(self.d["img"], self.img_off, self.H, self.W, self.stats, self.resized, self.dst_off)

    def vit(self):
        P.pace_vit_attn_importance(self.d["vit_q"], self.d["vit_k"], self.cu_patches,
                                   1.0 / math.sqrt(synth.VIT_DIM), 4, out=self.s_vis, ws=self.ws_vit)

    def llm(self):
        P.pace_llm_text_visual_importance(self.d["llm_q"], self.d["llm_k"], self.cu_q, self.cu_vis,
                                          1.0 / math.sqrt(synth.LLM_DIM), out=self.s_llm, ws=self.ws_llm)

    def select(self):
        P.pace_ddae_select(self.s_llm, self.s_vis, self.cu_vis, self.cu_keep, s_final=self.s_final,
                           weights=self.weights, kept=self.kept)

    def gather(self):
        P.pace_gather(self.d["embed"], self.kept[: int(self.cu_keep[-1])], dst=self.rows)

    def step(self):
        for _, f in self.parts:
            f()

    # -- one step from host memory ---------------------------------------------------------------
    # Input tensors in the order the calls need them.  They are copied on a side stream and the
    # compute stream waits only for what its next call reads; the ViT query rows come in
    # VIT_CHUNKS pieces after the keys, and the row log-sum-exp pass takes each piece as it lands.
    COPY_GROUPS = (("img",), ("vit_k",), ("vit_q",), ("llm_q", "llm_k"), ("embed",))
    CALL_NEEDS = {"density": "img", "llm": "llm_k", "gather": "embed"}
    VIT_CHUNKS = 4

    def step_from_host(self, pinned: dict, out_host: dict, copy_stream: Optional[torch.cuda.Stream] = None):
        """Copies this step's inputs from pinned host tensors (keys as in `self.host`), runs the six
        calls, and copies the results named in `out_host` back to (pinned) host tensors.

        The host-to-device copies run on `copy_stream` in call order, so the ViT K/Q copy overlaps
        density and resampling, and the ViT row pass starts on the first query rows while the rest
        are still in flight; each call waits only for the inputs it reads.  The next step's copies
        wait for this step's calls to finish (the device input buffers are reused)."""
        main = torch.cuda.current_stream(self.dev)
        cs = copy_stream if copy_stream is not None else torch.cuda.Stream(self.dev)
        cs.wait_stream(main)        # the previous step's calls have read their inputs
        ready, q_ready = {}, []
        ends = P.vit_chunk_rows(self.cu_patches, self.VIT_CHUNKS)
        with torch.cuda.stream(cs):
            for group in self.COPY_GROUPS:
                if group == ("vit_q",):
                    r0 = 0
                    for r1 in ends:
                        self.d["vit_q"][r0:r1].copy_(pinned["vit_q"][r0:r1], non_blocking=True)
                        ev = torch.cuda.Event()
                        ev.record(cs)
                        q_ready.append(ev)
                        r0 = int(r1)
                    continue
                for k in group:
                    self.d[k].copy_(pinned[k], non_blocking=True)
                ev = torch.cuda.Event()
                ev.record(cs)
                ready[group[-1]] = ev
        for name, f in self.parts:
            if name == "vit":
                P.pace_vit_attn_importance_chunked(self.d["vit_q"], self.d["vit_k"], self.cu_patches, ends, q_ready,
                                                   1.0 / math.sqrt(synth.VIT_DIM), 4, out=self.s_vis, ws=self.ws_vit)
                continue
            if name in self.CALL_NEEDS:
                main.wait_event(ready[self.CALL_NEEDS[name]])
            f()
        for k, v in out_host.items():      # attribute name -> host tensor of the same shape
            v.copy_(getattr(self, k), non_blocking=True)

    # -- results on the host ---------------------------------------------------------------------
    def resized_images(self):
        st = P.stats_dict(self.stats[: self.B])
        flat = self.resized.cpu().numpy()
        return [flat[o:o + s["h_out"] * s["w_out"] * 3].reshape(s["h_out"], s["w_out"], 3)
                for o, s in zip(self.dst_off, st)]
