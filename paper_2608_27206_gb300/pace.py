"""Thin ctypes binding of libpace (include/pace.h).

Every function here only marshals arguments: torch CUDA tensors become device
pointers, host index arrays become int32/int64 buffers, and the call goes to the
C ABI of the same name.  PyTorch supplies device memory and the current stream;
all arithmetic runs in the library's CUDA kernels.  If libpace.so has not been
built, the first call raises: there is no fallback path.
"""
from __future__ import annotations

import ctypes
import os
from typing import Optional, Sequence

import numpy as np
import torch

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "libpace.so")

PACE_OK, PACE_ERR_INVALID_ARG, PACE_ERR_UNSUPPORTED_ARCH = 0, 1, 2
PACE_ERR_WORKSPACE, PACE_ERR_CUDA, PACE_ERR_TIMEOUT = 3, 4, 5
STATS_FIELDS = ("phi", "rho_g", "d_top", "rho_d", "rho", "r", "n_patches", "k_tail", "h_out", "w_out")


class PaceError(RuntimeError):
    def __init__(self, fn: str, status: int, detail: str = ""):
        self.status = status
        super().__init__(f"{fn} failed: {status_string(status)}{detail}")


class ApcParams(ctypes.Structure):
    _fields_ = [("alpha", ctypes.c_float), ("gamma", ctypes.c_float), ("tail_frac", ctypes.c_float),
                ("r_min", ctypes.c_float), ("r_max", ctypes.c_float), ("align", ctypes.c_int32)]


class DdaeParams(ctypes.Structure):
    _fields_ = [("tau", ctypes.c_float), ("fusion", ctypes.c_int32)]


# fusion modes of DdaeParams (pace_ddae_fusion)
DDAE_ADAPTIVE, DDAE_ONLY_LLM, DDAE_ONLY_VIT, DDAE_FIXED = 0, 1, 2, 3
FEATURE_RGB_STATS, FEATURE_COLOR_ENTROPY, FEATURE_EDGE_DENSITY, FEATURE_LAPLACIAN = 0, 1, 2, 3
PIXEL_FEATURES = {"rgb_stats": 0, "color_entropy": 1, "edge_density": 2, "laplacian": 3}
PIXEL_FEATURE_DIM = 8   # floats per feature token (zero-padded)
QUERY_VISION_TEXT, QUERY_TEXT, QUERY_LAST = 0, 1, 2
QUERY_SETS = {"vision_text": QUERY_VISION_TEXT, "text": QUERY_TEXT, "last": QUERY_LAST}


class GatherTensor(ctypes.Structure):
    _fields_ = [("src", ctypes.c_void_p), ("dst", ctypes.c_void_p), ("row_bytes", ctypes.c_int64),
                ("src_row_stride", ctypes.c_int64), ("dst_row_stride", ctypes.c_int64), ("n_slabs", ctypes.c_int64),
                ("src_slab_stride", ctypes.c_int64), ("dst_slab_stride", ctypes.c_int64),
                ("n_src_rows", ctypes.c_int64)]


GATHER_MAX_TENSORS = 16


_P = ctypes.c_void_p
_I32P = ctypes.POINTER(ctypes.c_int32)
_I64P = ctypes.POINTER(ctypes.c_int64)
_SIGS = {
    "pace_status_string": (ctypes.c_char_p, [ctypes.c_int]),
    "pace_last_cuda_error": (ctypes.c_int, []),
    "pace_kernel_launch_count": (ctypes.c_uint64, []),
    "pace_selftest_wait_timeout": (ctypes.c_int, [ctypes.c_uint32, _P]),
    "pace_init": (ctypes.c_int, [ctypes.c_int]),
    "pace_device_status": (ctypes.c_int, [_I32P, _I32P, ctypes.c_int]),
    "pace_apc_params_default": (None, [ctypes.POINTER(ApcParams)]),
    "pace_apc_density_workspace_size": (ctypes.c_size_t, [ctypes.c_int, _I32P, _I32P]),
    "pace_budget_vanilla": (ctypes.c_int32, [ctypes.c_int32, ctypes.c_int32, ctypes.c_double]),
    "pace_prune_index": (ctypes.c_int, [ctypes.c_int, _I32P, _I32P, _I32P, _I32P, _P, _P, _P]),
    "pace_gather_multi": (ctypes.c_int, [ctypes.POINTER(GatherTensor), ctypes.c_int, _P, ctypes.c_int64, _P]),
    "pace_apc_density_tokens_workspace_size": (ctypes.c_size_t, [ctypes.c_int, _I32P, ctypes.c_int]),
    "pace_apc_density_tokens": (ctypes.c_int, [_P, _I32P, ctypes.c_int, ctypes.c_int, _I32P, _I32P,
                                               ctypes.POINTER(ApcParams), _P, _P, _P, ctypes.c_size_t, _P]),
    "pace_apc_density": (ctypes.c_int, [_P, _I64P, _I32P, _I32P, ctypes.c_int, ctypes.POINTER(ApcParams), _P, _P,
                                        _P, ctypes.c_size_t, _P]),
    "pace_apc_pixel_features": (ctypes.c_int, [_P, _I64P, _I32P, _I32P, ctypes.c_int, ctypes.c_int, _P, _P]),
    "pace_apc_density_pixel_workspace_size": (ctypes.c_size_t, [ctypes.c_int, _I32P, _I32P]),
    "pace_apc_density_pixel": (ctypes.c_int, [_P, _I64P, _I32P, _I32P, ctypes.c_int, ctypes.c_int,
                                              ctypes.POINTER(ApcParams), _P, _P, _P, ctypes.c_size_t, _P]),
    "pace_apc_density_static": (ctypes.c_int, [_P, _I64P, _I32P, _I32P, ctypes.c_int, ctypes.POINTER(ApcParams),
                                               _P, _P, _P]),
    "pace_apc_resample": (ctypes.c_int, [_P, _I64P, _I32P, _I32P, _P, _P, _I64P, ctypes.c_int, _P]),
    "pace_apc_resample_to": (ctypes.c_int, [_P, _I64P, _I32P, _I32P, _I32P, _I32P, _P, _I64P, ctypes.c_int, _P]),
    "pace_vit_attn_importance_workspace_size": (ctypes.c_size_t, [ctypes.c_int, _I32P, ctypes.c_int]),
    "pace_vit_attn_importance": (ctypes.c_int, [_P, _P, _I32P, ctypes.c_int, ctypes.c_int, ctypes.c_int,
                                                ctypes.c_float, ctypes.c_int, _P, _P, ctypes.c_size_t, _P]),
    "pace_vit_attn_importance_chunked": (ctypes.c_int, [_P, _P, _I32P, ctypes.c_int, ctypes.c_int, ctypes.c_int,
                                                        ctypes.c_float, ctypes.c_int, _P, _P, ctypes.c_size_t,
                                                        ctypes.c_int, _I64P, ctypes.POINTER(ctypes.c_void_p), _P]),
    "pace_llm_text_visual_importance_workspace_size": (ctypes.c_size_t, [ctypes.c_int, _I32P, _I32P, ctypes.c_int,
                                                                         ctypes.c_int]),
    "pace_llm_text_visual_importance": (ctypes.c_int, [_P, _P, _I32P, _I32P, ctypes.c_int, ctypes.c_int,
                                                       ctypes.c_int, ctypes.c_int, ctypes.c_float, _P, _P,
                                                       ctypes.c_size_t, _P]),
    "pace_llm_sequence_importance_workspace_size": (ctypes.c_size_t, [ctypes.c_int, _I32P, _I32P, _I32P,
                                                                      ctypes.c_int, ctypes.c_int, ctypes.c_int]),
    "pace_llm_sequence_importance": (ctypes.c_int, [_P, _P, _I32P, _I32P, _I32P, ctypes.c_int, ctypes.c_int,
                                                    ctypes.c_int, ctypes.c_int, ctypes.c_float, ctypes.c_int, _P,
                                                    _P, ctypes.c_size_t, _P]),
    "pace_ddae_params_default": (None, [ctypes.POINTER(DdaeParams)]),
    "pace_budget": (ctypes.c_int32, [ctypes.c_int32, ctypes.c_double]),
    "pace_ddae_select": (ctypes.c_int, [_P, _P, _I32P, _I32P, ctypes.c_int, ctypes.POINTER(DdaeParams), _P, _P,
                                        _P, _P]),
    "pace_gather": (ctypes.c_int, [_P, ctypes.c_int64, ctypes.c_int64, _P, ctypes.c_int64, _P, _P]),
}

_lib = None


def lib() -> ctypes.CDLL:
    """Opens libpace.so (once).  Raises if it is missing."""
    global _lib
    if _lib is None:
        if not os.path.exists(LIB_PATH):
            raise RuntimeError(f"{LIB_PATH} is not built; run paper_2608_27206_gb300.build.build() "
                               "(needs nvcc with sm_103a support)")
        L = ctypes.CDLL(LIB_PATH)
        for name, (res, args) in _SIGS.items():
            f = getattr(L, name)
            f.restype = res
            f.argtypes = args
        _lib = L
    return _lib


def status_string(status: int) -> str:
    return lib().pace_status_string(int(status)).decode()


def _check(fn: str, status: int):
    if status != PACE_OK:
        detail = f" (cudaError {lib().pace_last_cuda_error()})" if status == PACE_ERR_CUDA else ""
        raise PaceError(fn, status, detail)


def _i32(a) -> np.ndarray:
    return np.ascontiguousarray(np.asarray(a, dtype=np.int32))


def _i64(a) -> np.ndarray:
    return np.ascontiguousarray(np.asarray(a, dtype=np.int64))


def _pi32(a: np.ndarray):
    return a.ctypes.data_as(_I32P)


def _pi64(a: np.ndarray):
    return a.ctypes.data_as(_I64P)


def _dev(t: Optional[torch.Tensor]):
    if t is None:
        return None
    if not t.is_cuda:
        raise ValueError("expected a CUDA tensor")
    if not t.is_contiguous():
        raise ValueError("expected a contiguous tensor")
    return ctypes.c_void_p(t.data_ptr())


def _stream(stream):
    if stream is None:
        stream = torch.cuda.current_stream()
    return ctypes.c_void_p(stream.cuda_stream)


def _workspace(nbytes: int, ws: Optional[torch.Tensor], device) -> torch.Tensor:
    if ws is not None:
        if ws.numel() * ws.element_size() < nbytes:
            raise PaceError("workspace", PACE_ERR_WORKSPACE)
        return ws
    return torch.empty(max(int(nbytes), 16), dtype=torch.uint8, device=device)


# ----------------------------------------------------------------------------------------------
# library state
# ----------------------------------------------------------------------------------------------
def pace_init(device: int = 0) -> None:
    _check("pace_init", lib().pace_init(int(device)))


def pace_device_status(clear: bool = True):
    """(code, kernel id) of the device status word; synchronises the device."""
    code, where = ctypes.c_int32(0), ctypes.c_int32(0)
    _check("pace_device_status", lib().pace_device_status(ctypes.byref(code), ctypes.byref(where), int(clear)))
    return code.value, where.value


def pace_selftest_wait_timeout(limit_us: int, stream=None) -> None:
    """Launches a kernel whose bounded wait must run out and report PACE_ERR_TIMEOUT."""
    _check("pace_selftest_wait_timeout", lib().pace_selftest_wait_timeout(int(limit_us), _stream(stream)))


def pace_kernel_launch_count() -> int:
    """Kernels launched by libpace so far in this process."""
    return int(lib().pace_kernel_launch_count())


def pace_budget(n_vis: int, frac: float) -> int:
    return int(lib().pace_budget(int(n_vis), float(frac)))


def apc_params(**kw) -> ApcParams:
    p = ApcParams()
    lib().pace_apc_params_default(ctypes.byref(p))
    for k, v in kw.items():
        setattr(p, k, v)
    return p


def ddae_params(**kw) -> DdaeParams:
    p = DdaeParams()
    lib().pace_ddae_params_default(ctypes.byref(p))
    for k, v in kw.items():
        setattr(p, k, v)
    return p


# ----------------------------------------------------------------------------------------------
# Condense
# ----------------------------------------------------------------------------------------------
def pace_apc_density_workspace_size(H: Sequence[int], W: Sequence[int]) -> int:
    h, w = _i32(H), _i32(W)
    return int(lib().pace_apc_density_workspace_size(len(h), _pi32(h), _pi32(w)))


def pace_apc_density(img: torch.Tensor, img_off, H, W, params: Optional[ApcParams] = None,
                     d_out: Optional[torch.Tensor] = None, stats: Optional[torch.Tensor] = None,
                     ws: Optional[torch.Tensor] = None, stream=None):
    """APC density of B packed uint8 images.  Returns (d [sum N] float32, stats [B, 10] int32 view)."""
    off, h, w = _i64(img_off), _i32(H), _i32(W)
    B = len(h)
    n = int(((h // 14).astype(np.int64) * (w // 14)).sum())
    dev = img.device
    if d_out is None:
        d_out = torch.empty(max(n, 1), dtype=torch.float32, device=dev)
    if stats is None:
        stats = torch.zeros((max(B, 1), 10), dtype=torch.int32, device=dev)
    nbytes = pace_apc_density_workspace_size(h, w)
    ws = _workspace(nbytes, ws, dev)
    st = lib().pace_apc_density(_dev(img), _pi64(off), _pi32(h), _pi32(w), B,
                                ctypes.byref(params) if params is not None else None, _dev(d_out), _dev(stats),
                                _dev(ws), ws.numel() * ws.element_size(), _stream(stream))
    _check("pace_apc_density", st)
    return d_out[:n], stats[:B]


def _feature(feature) -> int:
    return PIXEL_FEATURES[feature] if isinstance(feature, str) else int(feature)


def pace_apc_pixel_features(img: torch.Tensor, img_off, H, W, feature, out: Optional[torch.Tensor] = None,
                            stream=None) -> torch.Tensor:
    """Pixel-statistic feature tokens float32 [sum N, 8] of B packed uint8 images; feature is
    "rgb_stats", "color_entropy", "edge_density", "laplacian" or a FEATURE_* code."""
    off, h, w = _i64(img_off), _i32(H), _i32(W)
    B = len(h)
    n = int(((h // 14).astype(np.int64) * (w // 14)).sum())
    if out is None:
        out = torch.empty((max(n, 1), PIXEL_FEATURE_DIM), dtype=torch.float32, device=img.device)
    st = lib().pace_apc_pixel_features(_dev(img), _pi64(off), _pi32(h), _pi32(w), B, _feature(feature), _dev(out),
                                       _stream(stream))
    _check("pace_apc_pixel_features", st)
    return out[:n]


def pace_apc_density_pixel_workspace_size(H, W) -> int:
    h, w = _i32(H), _i32(W)
    return int(lib().pace_apc_density_pixel_workspace_size(len(h), _pi32(h), _pi32(w)))


def pace_apc_density_pixel(img: torch.Tensor, img_off, H, W, feature, params: Optional[ApcParams] = None,
                           d_out: Optional[torch.Tensor] = None, stats: Optional[torch.Tensor] = None,
                           ws: Optional[torch.Tensor] = None, stream=None):
    """APC density with a pixel-statistic preview.  Returns (d [sum N], stats [B, 10])."""
    off, h, w = _i64(img_off), _i32(H), _i32(W)
    B = len(h)
    n = int(((h // 14).astype(np.int64) * (w // 14)).sum())
    dev = img.device
    if d_out is None:
        d_out = torch.empty(max(n, 1), dtype=torch.float32, device=dev)
    if stats is None:
        stats = torch.zeros((max(B, 1), 10), dtype=torch.int32, device=dev)
    ws = _workspace(pace_apc_density_pixel_workspace_size(h, w), ws, dev)
    st = lib().pace_apc_density_pixel(_dev(img), _pi64(off), _pi32(h), _pi32(w), B, _feature(feature),
                                      ctypes.byref(params) if params is not None else None, _dev(d_out), _dev(stats),
                                      _dev(ws), ws.numel() * ws.element_size(), _stream(stream))
    _check("pace_apc_density_pixel", st)
    return d_out[:n], stats[:B]


PACE_APC_STATIC_MAX_IMAGES = 16
PACE_APC_STATIC_MAX_PATCHES = 65536


def pace_apc_density_static(img: torch.Tensor, img_off, H, W, params: Optional[ApcParams] = None,
                            d_out: Optional[torch.Tensor] = None, stats: Optional[torch.Tensor] = None,
                            stream=None):
    """pace_apc_density with the library's own static scratch: no workspace argument.

    For callers that cannot allocate device scratch.  Limited to PACE_APC_STATIC_MAX_IMAGES
    images and PACE_APC_STATIC_MAX_PATCHES patches per call; calls that overlap on the GPU
    share one scratch array and must be serialised.  Returns (d, stats) like pace_apc_density.
    """
    off, h, w = _i64(img_off), _i32(H), _i32(W)
    B = len(h)
    n = int(((h // 14).astype(np.int64) * (w // 14)).sum())
    dev = img.device
    if d_out is None:
        d_out = torch.empty(max(n, 1), dtype=torch.float32, device=dev)
    if stats is None:
        stats = torch.zeros((max(B, 1), 10), dtype=torch.int32, device=dev)
    st = lib().pace_apc_density_static(_dev(img), _pi64(off), _pi32(h), _pi32(w), B,
                                       ctypes.byref(params) if params is not None else None, _dev(d_out),
                                       _dev(stats), _stream(stream))
    _check("pace_apc_density_static", st)
    return d_out[:n], stats[:B]


def pace_apc_density_tokens_workspace_size(cu_tokens, D: int) -> int:
    cu = _i32(cu_tokens)
    return int(lib().pace_apc_density_tokens_workspace_size(len(cu) - 1, _pi32(cu), D))


def pace_apc_density_tokens(T: torch.Tensor, cu_tokens, H, W, params: Optional[ApcParams] = None,
                            d_out: Optional[torch.Tensor] = None, stats: Optional[torch.Tensor] = None,
                            ws: Optional[torch.Tensor] = None, stream=None):
    """APC density of B images' preview tokens T (bf16 [sum N, D]).  Returns (d [sum N], stats)."""
    cu, h, w = _i32(cu_tokens), _i32(H), _i32(W)
    B = len(cu) - 1
    n, D = int(cu[-1]), int(T.shape[-1])
    dev = T.device
    if d_out is None:
        d_out = torch.empty(max(n, 1), dtype=torch.float32, device=dev)
    if stats is None:
        stats = torch.zeros((max(B, 1), 10), dtype=torch.int32, device=dev)
    if ws is None:
        ws = torch.empty(max(pace_apc_density_tokens_workspace_size(cu, D), 16), dtype=torch.uint8, device=dev)
    st = lib().pace_apc_density_tokens(_dev(T), _pi32(cu), B, D, _pi32(h), _pi32(w),
                                       ctypes.byref(params) if params is not None else None, _dev(d_out),
                                       _dev(stats), _dev(ws), ws.numel(), _stream(stream))
    _check("pace_apc_density_tokens", st)
    return d_out[:n], stats[:B]


def pace_budget_vanilla(n_vis_vanilla: int, n_vis_condensed: int, frac: float) -> int:
    return int(lib().pace_budget_vanilla(int(n_vis_vanilla), int(n_vis_condensed), float(frac)))


def pace_prune_index(cu_seq, vis_start, cu_vis, cu_keep, kept: torch.Tensor, out: Optional[torch.Tensor] = None,
                     stream=None):
    """Row list of the pruned sequences (global pre-prune rows), int32 on kept's device."""
    sq, vs, v, kp = _i32(cu_seq), _i32(vis_start), _i32(cu_vis), _i32(cu_keep)
    B = len(sq) - 1
    n_out = int((sq[1:] - sq[:-1]).sum() - v[-1] + kp[-1]) if B > 0 else 0
    if out is None:
        out = torch.empty(max(n_out, 1), dtype=torch.int32, device=kept.device)
    st = lib().pace_prune_index(B, _pi32(sq), _pi32(vs), _pi32(v), _pi32(kp), _dev(kept), _dev(out), _stream(stream))
    _check("pace_prune_index", st)
    return out[:n_out]


def gather_spec(src: torch.Tensor, dst: torch.Tensor, dim: int) -> GatherTensor:
    """Descriptor for gathering contiguous src along `dim` into contiguous dst: the dimensions
    before `dim` are slabs, the ones after it form a row."""
    if not (src.is_contiguous() and dst.is_contiguous()) or src.dtype != dst.dtype:
        raise ValueError("gather_spec needs contiguous src and dst of one dtype")
    if src.shape[:dim] != dst.shape[:dim] or src.shape[dim + 1:] != dst.shape[dim + 1:]:
        raise ValueError("src and dst may differ only along the gathered dimension")
    es = src.element_size()
    row = es * int(np.prod(src.shape[dim + 1:], dtype=np.int64))
    slabs = int(np.prod(src.shape[:dim], dtype=np.int64))
    return GatherTensor(src.data_ptr(), dst.data_ptr(), row, row, row, slabs, row * src.shape[dim],
                        row * dst.shape[dim], src.shape[dim])


def pace_gather_multi(specs, idx: torch.Tensor, stream=None):
    """Gathers every GatherTensor in `specs` with the same row list idx (device int32)."""
    arr = (GatherTensor * max(len(specs), 1))(*specs)
    st = lib().pace_gather_multi(arr, len(specs), _dev(idx), idx.numel(), _stream(stream))
    _check("pace_gather_multi", st)


def stats_dict(stats: torch.Tensor):
    """Decodes pace_apc_stats rows ([B, 10] int32) into a list of dicts."""
    a = stats.detach().cpu().numpy().astype(np.int32)
    f = a.view(np.float32)
    out = []
    for i in range(a.shape[0]):
        d = {k: float(f[i, j]) for j, k in enumerate(STATS_FIELDS[:6])}
        d.update({k: int(a[i, 6 + j]) for j, k in enumerate(STATS_FIELDS[6:])})
        out.append(d)
    return out


def pace_apc_resample(src: torch.Tensor, src_off, H, W, stats: torch.Tensor, dst: torch.Tensor, dst_off,
                      stream=None) -> None:
    off, h, w, doff = _i64(src_off), _i32(H), _i32(W), _i64(dst_off)
    _check("pace_apc_resample", lib().pace_apc_resample(_dev(src), _pi64(off), _pi32(h), _pi32(w), _dev(stats),
                                                        _dev(dst), _pi64(doff), len(h), _stream(stream)))


def pace_apc_resample_to(src: torch.Tensor, src_off, H, W, H_out, W_out, dst: torch.Tensor, dst_off,
                         stream=None) -> None:
    off, h, w, doff = _i64(src_off), _i32(H), _i32(W), _i64(dst_off)
    ho, wo = _i32(H_out), _i32(W_out)
    _check("pace_apc_resample_to", lib().pace_apc_resample_to(_dev(src), _pi64(off), _pi32(h), _pi32(w), _pi32(ho),
                                                              _pi32(wo), _dev(dst), _pi64(doff), len(h),
                                                              _stream(stream)))


# ----------------------------------------------------------------------------------------------
# Extract
# ----------------------------------------------------------------------------------------------
def pace_vit_attn_importance_workspace_size(cu_seqlens, n_heads: int) -> int:
    cu = _i32(cu_seqlens)
    return int(lib().pace_vit_attn_importance_workspace_size(len(cu) - 1, _pi32(cu), int(n_heads)))


def pace_vit_attn_importance(Q: torch.Tensor, K: torch.Tensor, cu_seqlens, scale: Optional[float] = None,
                             merge: int = 4, out: Optional[torch.Tensor] = None,
                             ws: Optional[torch.Tensor] = None, stream=None) -> torch.Tensor:
    """S_vis_raw [total / merge] from bf16 Q, K [total, heads, head_dim]."""
    cu = _i32(cu_seqlens)
    B = len(cu) - 1
    total, Hh, D = Q.shape
    if scale is None:
        scale = float(D) ** -0.5
    if out is None:
        out = torch.empty(max(int(cu[-1]) // merge, 1), dtype=torch.float32, device=Q.device)
    ws = _workspace(pace_vit_attn_importance_workspace_size(cu, Hh), ws, Q.device)
    st = lib().pace_vit_attn_importance(_dev(Q), _dev(K), _pi32(cu), B, Hh, D, float(scale), int(merge), _dev(out),
                                        _dev(ws), ws.numel() * ws.element_size(), _stream(stream))
    _check("pace_vit_attn_importance", st)
    return out[: int(cu[-1]) // merge]


def vit_chunk_rows(cu_seqlens, n_chunks: int, pair: int = 256) -> np.ndarray:
    """End rows of `n_chunks` near-equal pieces of Q, each end moved down to the end of a
    `pair`-row block of its image (or the image's end), so no block waits for a later piece."""
    cu = _i32(cu_seqlens).astype(np.int64)
    total = int(cu[-1])
    ends = []
    for c in range(1, n_chunks):
        r = total * c // n_chunks
        b = int(np.searchsorted(cu, r, side="right")) - 1
        b = min(max(b, 0), len(cu) - 2)
        e = int(cu[b]) + (r - int(cu[b])) // pair * pair
        ends.append(max(e, ends[-1] if ends else 0))
    ends.append(total)
    return np.asarray(ends, dtype=np.int64)


def pace_vit_attn_importance_chunked(Q: torch.Tensor, K: torch.Tensor, cu_seqlens, chunk_end_rows,
                                     chunk_ready: Sequence[torch.cuda.Event], scale: Optional[float] = None,
                                     merge: int = 4, out: Optional[torch.Tensor] = None,
                                     ws: Optional[torch.Tensor] = None, stream=None) -> torch.Tensor:
    """pace_vit_attn_importance whose row log-sum-exp pass runs in pieces of query rows, piece c
    after the (already recorded) event chunk_ready[c]; bit-identical results."""
    cu = _i32(cu_seqlens)
    B = len(cu) - 1
    total, Hh, D = Q.shape
    if scale is None:
        scale = float(D) ** -0.5
    if out is None:
        out = torch.empty(max(int(cu[-1]) // merge, 1), dtype=torch.float32, device=Q.device)
    ends = _i64(chunk_end_rows)
    if len(chunk_ready) != len(ends):
        raise ValueError("one event per chunk")
    evs = (ctypes.c_void_p * max(len(ends), 1))(*[int(e.cuda_event) for e in chunk_ready])
    ws = _workspace(pace_vit_attn_importance_workspace_size(cu, Hh), ws, Q.device)
    st = lib().pace_vit_attn_importance_chunked(_dev(Q), _dev(K), _pi32(cu), B, Hh, D, float(scale), int(merge),
                                                _dev(out), _dev(ws), ws.numel() * ws.element_size(), len(ends),
                                                _pi64(ends), evs, _stream(stream))
    _check("pace_vit_attn_importance_chunked", st)
    return out[: int(cu[-1]) // merge]


def pace_llm_text_visual_importance_workspace_size(cu_q, cu_k, n_q_heads: int, n_kv_heads: int) -> int:
    q, k = _i32(cu_q), _i32(cu_k)
    return int(lib().pace_llm_text_visual_importance_workspace_size(len(q) - 1, _pi32(q), _pi32(k), int(n_q_heads),
                                                                    int(n_kv_heads)))


def pace_llm_text_visual_importance(Q: torch.Tensor, K: torch.Tensor, cu_q, cu_k, scale: Optional[float] = None,
                                    out: Optional[torch.Tensor] = None, ws: Optional[torch.Tensor] = None,
                                    stream=None) -> torch.Tensor:
    """S_llm_raw [sum Nv] from bf16 Q [sum Tq, Hq, D] and K [sum Nv, Hkv, D]."""
    q, k = _i32(cu_q), _i32(cu_k)
    B = len(q) - 1
    _, Hq, D = Q.shape
    Hkv = K.shape[1]
    if scale is None:
        scale = float(D) ** -0.5
    if out is None:
        out = torch.empty(max(int(k[-1]), 1), dtype=torch.float32, device=Q.device)
    ws = _workspace(pace_llm_text_visual_importance_workspace_size(q, k, Hq, Hkv), ws, Q.device)
    st = lib().pace_llm_text_visual_importance(_dev(Q), _dev(K), _pi32(q), _pi32(k), B, Hq, Hkv, D, float(scale),
                                               _dev(out), _dev(ws), ws.numel() * ws.element_size(), _stream(stream))
    _check("pace_llm_text_visual_importance", st)
    return out[: int(k[-1])]


def _query_set(query_set) -> int:
    return QUERY_SETS[query_set] if isinstance(query_set, str) else int(query_set)


def pace_llm_sequence_importance_workspace_size(cu_seq, vis_start, n_vis, n_q_heads: int, n_kv_heads: int,
                                                query_set="vision_text") -> int:
    c, v, n = _i32(cu_seq), _i32(vis_start), _i32(n_vis)
    return int(lib().pace_llm_sequence_importance_workspace_size(len(c) - 1, _pi32(c), _pi32(v), _pi32(n),
                                                                 int(n_q_heads), int(n_kv_heads),
                                                                 _query_set(query_set)))


def pace_llm_sequence_importance(Q: torch.Tensor, K: torch.Tensor, cu_seq, vis_start, n_vis,
                                 query_set="vision_text", scale: Optional[float] = None,
                                 out: Optional[torch.Tensor] = None, ws: Optional[torch.Tensor] = None,
                                 stream=None) -> torch.Tensor:
    """Full-sequence S_llm_raw [sum n_vis] from bf16 Q [sum S, Hq, D] and K [sum S, Hkv, D] of causal
    sequences; query_set is "vision_text", "text" or "last" (or a QUERY_* code)."""
    c, v, n = _i32(cu_seq), _i32(vis_start), _i32(n_vis)
    B = len(c) - 1
    _, Hq, D = Q.shape
    Hkv = K.shape[1]
    qs = _query_set(query_set)
    if scale is None:
        scale = float(D) ** -0.5
    total = int(n.sum()) if B > 0 else 0
    if out is None:
        out = torch.empty(max(total, 1), dtype=torch.float32, device=Q.device)
    ws = _workspace(pace_llm_sequence_importance_workspace_size(c, v, n, Hq, Hkv, qs), ws, Q.device)
    st = lib().pace_llm_sequence_importance(_dev(Q), _dev(K), _pi32(c), _pi32(v), _pi32(n), B, Hq, Hkv, D,
                                            float(scale), qs, _dev(out), _dev(ws), ws.numel() * ws.element_size(),
                                            _stream(stream))
    _check("pace_llm_sequence_importance", st)
    return out[:total]


def pace_ddae_select(s_llm_raw: torch.Tensor, s_vis_raw: torch.Tensor, cu_v, cu_keep,
                     params: Optional[DdaeParams] = None, s_final: Optional[torch.Tensor] = None,
                     weights: Optional[torch.Tensor] = None, kept: Optional[torch.Tensor] = None, stream=None):
    """Returns (s_final [sum Nv], weights [B, 2], kept int32 [sum K])."""
    v, kp = _i32(cu_v), _i32(cu_keep)
    B = len(v) - 1
    dev = s_llm_raw.device
    if s_final is None:
        s_final = torch.empty(max(int(v[-1]), 1), dtype=torch.float32, device=dev)
    if weights is None:
        weights = torch.empty((max(B, 1), 2), dtype=torch.float32, device=dev)
    if kept is None:
        kept = torch.empty(max(int(kp[-1]), 1), dtype=torch.int32, device=dev)
    st = lib().pace_ddae_select(_dev(s_llm_raw), _dev(s_vis_raw), _pi32(v), _pi32(kp), B,
                                ctypes.byref(params) if params is not None else None, _dev(s_final),
                                _dev(weights), _dev(kept), _stream(stream))
    _check("pace_ddae_select", st)
    return s_final[: int(v[-1])], weights[:B], kept[: int(kp[-1])]


def pace_gather(src: torch.Tensor, idx: torch.Tensor, dst: Optional[torch.Tensor] = None, stream=None):
    """dst[r] = src[idx[r]] row by row (byte copy); src is [rows, ...] contiguous."""
    n_src = src.shape[0]
    row_bytes = src[0].numel() * src.element_size() if n_src else 0
    n = idx.numel()
    if dst is None:
        dst = torch.empty((max(n, 1),) + tuple(src.shape[1:]), dtype=src.dtype, device=src.device)
    st = lib().pace_gather(_dev(src), n_src, row_bytes, _dev(idx), n, _dev(dst), _stream(stream))
    _check("pace_gather", st)
    return dst[:n]
