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

    # -- the six calls (inputs from `d`, default: the resident copies) ---------------------------
    def density(self, d=None):
        d = d or self.d
        P.pace_apc_density(d["img"], self.img_off, self.H, self.W, d_out=self.dist, stats=self.stats,
                           ws=self.ws_density)

    def resample(self, d=None):
        d = d or self.d
        P.pace_apc_resample(d["img"], self.img_off, self.H, self.W, self.stats, self.resized, self.dst_off)

    def vit(self, d=None):
        d = d or self.d
        P.pace_vit_attn_importance(d["vit_q"], d["vit_k"], self.cu_patches,
                                   1.0 / math.sqrt(synth.VIT_DIM), 4, out=self.s_vis, ws=self.ws_vit)

    def llm(self, d=None):
        d = d or self.d
        P.pace_llm_text_visual_importance(d["llm_q"], d["llm_k"], self.cu_q, self.cu_vis,
                                          1.0 / math.sqrt(synth.LLM_DIM), out=self.s_llm, ws=self.ws_llm)

    def select(self, d=None):
        P.pace_ddae_select(self.s_llm, self.s_vis, self.cu_vis, self.cu_keep, s_final=self.s_final,
                           weights=self.weights, kept=self.kept)

    def gather(self, d=None):
        d = d or self.d
        P.pace_gather(d["embed"], self.kept[: int(self.cu_keep[-1])], dst=self.rows)

    def step(self):
        for _, f in self.parts:
            f()

    # -- one step from host memory ---------------------------------------------------------------
    # Input tensors in the order the calls need them.  They are copied on a side stream into one of
    # two device input slots, and the compute stream waits only for what its next call reads.
    COPY_GROUPS = (("img",), ("vit_k",), ("vit_q",), ("llm_q", "llm_k"), ("embed",))
    CALL_NEEDS = {"density": "img", "llm": "llm_k", "gather": "embed"}
    # which call overwrites each result that can be read back
    WRITERS = {"stats": "density", "dist": "density", "resized": "resample", "s_vis": "vit", "s_llm": "llm",
               "s_final": "select", "weights": "select", "kept": "select", "rows": "gather"}
    VIT_CHUNKS = 4

    def step_from_host(self, pinned: dict, out_host: dict, copy_stream: Optional[torch.cuda.Stream] = None,
                       readback_stream: Optional[torch.cuda.Stream] = None) -> torch.cuda.Event:
        """Copies this step's inputs from pinned host tensors (keys as in `self.host`), runs the six
        calls, and copies the results named in `out_host` back to (pinned) host tensors.  Returns
        the event after which those host tensors hold this step's results.

        Steps alternate between two device input slots: a step's copies wait only for the calls of
        the step before the previous one (the last reader of their slot), so while image n is being
        processed the inputs of image n + 1 are already crossing the host link, and the results of
        image n go back on `readback_stream` while image n + 1 is processed (a call that overwrites
        a result waits for its read-back).  Within a step the ViT K/Q copy overlaps density and
        resampling.  When nothing else is in flight (the previous step has finished), the ViT
        query rows are copied in VIT_CHUNKS pieces and the row log-sum-exp pass takes each piece
        as it lands; behind a running step the copy is done long before the ViT call, and one
        launch avoids the pieces' partial last waves."""
        main = torch.cuda.current_stream(self.dev)
        cs = copy_stream if copy_stream is not None else torch.cuda.Stream(self.dev)
        if not hasattr(self, "_slots"):
            self._slots = [self.d, {k: torch.empty_like(v) for k, v in self.d.items()}]
            self._slot_free = [None, None]
            self._slot_next = 0
            self._readback = {}
        rs = readback_stream if readback_stream is not None else torch.cuda.Stream(self.dev)
        si = self._slot_next
        self._slot_next ^= 1
        d = self._slots[si]
        prev = self._slot_free[si ^ 1]
        chunked = prev is None or prev.query()
        if self._slot_free[si] is not None:
            cs.wait_event(self._slot_free[si])      # the calls that last read this slot are done
        else:
            cs.wait_stream(main)
        ready, q_ready = {}, []
        ends = P.vit_chunk_rows(self.cu_patches, self.VIT_CHUNKS if chunked else 1)
        with torch.cuda.stream(cs):
            for group in self.COPY_GROUPS:
                if group == ("vit_q",):
                    r0 = 0
                    for r1 in ends:
                        d["vit_q"][r0:r1].copy_(pinned["vit_q"][r0:r1], non_blocking=True)
                        ev = torch.cuda.Event()
                        ev.record(cs)
                        q_ready.append(ev)
                        r0 = int(r1)
                    continue
                for k in group:
                    d[k].copy_(pinned[k], non_blocking=True)
                ev = torch.cuda.Event()
                ev.record(cs)
                ready[group[-1]] = ev
        for name, f in self.parts:
            if name in self._readback:
                main.wait_event(self._readback.pop(name))   # the previous results of this call are read
            if name == "vit":
                if chunked:
                    P.pace_vit_attn_importance_chunked(d["vit_q"], d["vit_k"], self.cu_patches, ends, q_ready,
                                                       1.0 / math.sqrt(synth.VIT_DIM), 4, out=self.s_vis,
                                                       ws=self.ws_vit)
                    continue
                main.wait_event(q_ready[-1])
            elif name in self.CALL_NEEDS:
                main.wait_event(ready[self.CALL_NEEDS[name]])
            f(d)
        free = torch.cuda.Event()
        free.record(main)
        self._slot_free[si] = free
        rs.wait_event(free)
        order = [k for name, _ in self.parts for k in out_host if self.WRITERS.get(k, "density") == name]
        done = free
        with torch.cuda.stream(rs):
            for k in order:     # in the order the next step overwrites them
                out_host[k].copy_(getattr(self, k), non_blocking=True)
                done = torch.cuda.Event()
                done.record(rs)
                self._readback[self.WRITERS.get(k, "density")] = done
        return done

    # -- results on the host ---------------------------------------------------------------------
    def resized_images(self):
        st = P.stats_dict(self.stats[: self.B])
        flat = self.resized.cpu().numpy()
        return [flat[o:o + s["h_out"] * s["w_out"] * 3].reshape(s["h_out"], s["w_out"], 3)
                for o, s in zip(self.dst_off, st)]
