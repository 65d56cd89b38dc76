"""fp64 CPU oracle for PACE's condense-and-extract hot path.

TEST INFRASTRUCTURE ONLY.  Only the tests, ``__graft_entry__.smoke()`` and the
CPU-baseline leg of ``bench.py`` may import this module.  The product path (the
CUDA library and its binding) never reads it, and it shares no code with them.

Every function is a plain, slow statement of one step of the method, written
from the paper (arxiv 2608.27206, "PACE: A Unified Condense-and-Extract
Paradigm for Fast VLM Inference"), in float64, with numpy library primitives
(matmul, sort, exp) as the only building blocks.  Citations name the paper's
sections and equations.

Readings taken where the paper is silent or cannot be followed literally
(each is listed again, with its reason, in the design notes):
  R1  APC preview feature: the paper's T_v is the output of ViT block 1
      (Sec. 3.2, "Shallow Feature Preview").  No ViT weights are used here, so
      the token of patch i is the stand-in T_i = [x_i / 255 ; 1], x_i the
      14x14x3 patch in (row, column, channel) order, patches in raster order.
  R2  "top 10 %" of d_i: k_tail = max(1, floor(tail_frac * N + 0.5)).
  R3  r = min(max(rho, r_min), r_max); r_max is the hard budget cap of
      Sec. 3.2 "Adaptive Condensation" (default 1, i.e. no cap), r_min = 0.
  R4  target size: both sides scaled by sqrt(r) (App. B.3) and snapped to the
      28-pixel merge unit: H' = min(H, max(28, 28 * floor(H sqrt(r) / 28 + 0.5))).
  R5  bicubic resize: separable cubic convolution (a = -0.5), centre-aligned
      sampling, support widened by the downscale factor (antialias), window
      clipped at the border, weights renormalised; round half to even.
  R6  S_vis: the attention each patch receives in the final ViT block, summed
      over heads and query rows (softmax over all patches of the image, no
      mask), then summed over the 4 patches of each 2x2 merge unit.
  R7  S_llm: text queries over the visual keys only (no mask), GQA head
      h -> KV head h // (Hq / Hkv), summed over heads and queries.
  R8  min-max of a constant map gives 0; sigma is the population deviation.
  R9  top-K ties: the lower index wins; the kept indices are returned in
      ascending order.  K = floor(p * N_vis + 0.5) clamped to [0, N_vis].
  R10 preview tokens given by the caller (apc_density_preview): a token of zero
      norm counts as t_hat = 0 (cosine 0 with every token, Eq. 1 undefined
      otherwise); if every token is zero, c_hat = 0.
  R11 full-sequence S_llm (llm_sequence_importance): the query set starts at
      the first visual position (Vision + Text; earlier positions cannot see
      the visual span under the causal mask), after the visual span (Text) or
      at the last position (Last); each query's softmax runs over every
      position up to and including itself.
  R14 pixel-statistic preview features (pixel_statistic_tokens; App. "Shallow
      Feature Preview Ablation" names them without a definition): per 14x14
      patch, with luma Y' = 299 R + 587 G + 114 B in integers (BT.601 weights
      in thousandths; Y = Y' / 255000 in [0, 1]) and the patch's 12x12 interior
      for the 3x3 operators:
        rgb_stats      [mean_R, mean_G, mean_B, std_R, std_G, std_B, 1] of x / 255
                       (population standard deviations);
        color_entropy  [H_R, H_G, H_B, 4] / 4, H_c the Shannon entropy (bits) of
                       the patch's 16-bin histogram of channel c (bin = value >> 4);
        edge_density   [e, 1], e the fraction of interior pixels whose Sobel
                       gradient magnitude of Y exceeds 0.25;
        laplacian      [s, 1], s the population standard deviation of the
                       4-neighbour Laplacian of Y over the interior.
      The constant last coordinate plays the role it has in R1: a token is never
      zero and the cosines of Eq. 1 see the size of the statistic.
"""
from __future__ import annotations

import math
from typing import Dict, List, Sequence

import numpy as np

PATCH = 14
MERGE_UNIT = 28

# Hyper-parameters the paper fixes (Sec. 4.1 "Implementation Details", App. B.3).
ALPHA = 0.6      # global/local balance of Eq. 6
GAMMA = 1.5      # local contrast scaling of Eq. 5
TAIL_FRAC = 0.10  # "top 10 %" tail of d_i (Sec. 3.2; App. tail-percentile study)
TAU = 0.5        # fusion temperature of Eq. 7


# ==============================================================================================
# Condense: Adaptive Pixel Compressor (Sec. 3.2)
# ==============================================================================================
def patch_tokens(img: np.ndarray) -> np.ndarray:
    """Reading R1: stand-in preview tokens T [N, 589] of a uint8 HxWx3 image."""
    H, W, _ = img.shape
    gh, gw = H // PATCH, W // PATCH
    x = img[: gh * PATCH, : gw * PATCH].astype(np.float64) / 255.0
    x = x.reshape(gh, PATCH, gw, PATCH, 3).transpose(0, 2, 1, 3, 4).reshape(gh * gw, PATCH * PATCH * 3)
    return np.concatenate([x, np.ones((gh * gw, 1))], axis=1)


def unit_rows(T: np.ndarray) -> np.ndarray:
    """l2-normalised rows; a zero row stays zero (reading R10: its cosine with any token is 0)."""
    nrm = np.linalg.norm(T, axis=1, keepdims=True)
    return np.divide(T, nrm, out=np.zeros_like(T, dtype=np.float64), where=nrm > 0)


def global_redundancy(T: np.ndarray, rows_per_block: int = 512) -> float:
    """Eq. 1: phi = (1/N^2) sum_i sum_j cos(T_i, T_j), summed literally over all N^2 pairs."""
    Tn = unit_rows(T)
    N = Tn.shape[0]
    total = 0.0
    for i0 in range(0, N, rows_per_block):
        total += float((Tn[i0:i0 + rows_per_block] @ Tn.T).sum())
    return total / (N * N)


def apc_density_tokens(T: np.ndarray, alpha: float = ALPHA, gamma: float = GAMMA,
                       tail_frac: float = TAIL_FRAC) -> Dict[str, object]:
    """Eq. 1-6 on preview tokens T [N, D] (any N >= 1, any D)."""
    N = T.shape[0]
    Tn = unit_rows(T)                                           # l2-normalised tokens
    phi = global_redundancy(T)                                  # Eq. 1
    rho_g = 1.0 - phi                                           # Eq. 2
    c = Tn.mean(axis=0)                                         # Eq. 3
    cn = np.linalg.norm(c)
    c_hat = c / cn if cn > 0 else np.zeros_like(c)              # reading R10
    d = np.linalg.norm(Tn - c_hat[None, :], axis=1)             # Eq. 4
    k_tail = max(1, int(math.floor(tail_frac * N + 0.5)))       # reading R2
    d_top = float(np.sort(d)[::-1][:k_tail].mean())
    rho_d = min(d_top / gamma, 1.0)                             # Eq. 5
    rho = alpha * rho_g + (1.0 - alpha) * rho_d                 # Eq. 6
    return dict(N=N, phi=phi, rho_g=rho_g, c=c, c_hat=c_hat, d=d, k_tail=k_tail,
                d_top=d_top, rho_d=rho_d, rho=rho)


def apc_density_preview(T: np.ndarray, H: int, W: int, alpha: float = ALPHA, gamma: float = GAMMA,
                        tail_frac: float = TAIL_FRAC, r_min: float = 0.0, r_max: float = 1.0):
    """Sec. 3.2 on the paper's own input: preview tokens T [N, D] of an H x W image."""
    st = apc_density_tokens(np.asarray(T, dtype=np.float64), alpha, gamma, tail_frac)
    st["r"] = retention_ratio(st["rho"], r_min, r_max)
    st["H_out"], st["W_out"] = target_size(H, W, st["r"])
    return st


def retention_ratio(rho: float, r_min: float = 0.0, r_max: float = 1.0) -> float:
    """Sec. 3.2 'Adaptive Condensation': r = rho, capped by the budget's maximum ratio (R3)."""
    return min(max(rho, r_min), r_max)


def target_size(H: int, W: int, r: float):
    """App. B.3: width and height scaled by sqrt(r), snapped to 28 px (reading R4)."""
    s = math.sqrt(max(r, 0.0))

    def side(n):
        return min(n, max(MERGE_UNIT, MERGE_UNIT * int(math.floor(n * s / MERGE_UNIT + 0.5))))
    return side(H), side(W)


def apc_density(img: np.ndarray, alpha: float = ALPHA, gamma: float = GAMMA,
                tail_frac: float = TAIL_FRAC, r_min: float = 0.0, r_max: float = 1.0):
    """Full APC decision for one image: density statistics, r and the target size."""
    st = apc_density_tokens(patch_tokens(img), alpha, gamma, tail_frac)
    st["r"] = retention_ratio(st["rho"], r_min, r_max)
    st["H_out"], st["W_out"] = target_size(img.shape[0], img.shape[1], st["r"])
    return st


# Pixel-statistic preview features (App. "Shallow Feature Preview Ablation"), reading R14.
PIXEL_FEATURES = ("rgb_stats", "color_entropy", "edge_density", "laplacian")
FEATURE_DIMS = {"rgb_stats": 7, "color_entropy": 4, "edge_density": 2, "laplacian": 2}
LUMA_WEIGHTS = (299, 587, 114)   # thousandths; Y' = 299 R + 587 G + 114 B
LUMA_SCALE = 255000              # Y' of a white pixel
EDGE_TAU = 0.25                  # Sobel magnitude threshold on Y in [0, 1]
ENTROPY_BINS = 16


def patches(img: np.ndarray) -> np.ndarray:
    """The 14x14x3 patches of an image in raster order: uint8 [N, 14, 14, 3]."""
    H, W, _ = img.shape
    gh, gw = H // PATCH, W // PATCH
    x = img[: gh * PATCH, : gw * PATCH]
    return x.reshape(gh, PATCH, gw, PATCH, 3).transpose(0, 2, 1, 3, 4).reshape(gh * gw, PATCH, PATCH, 3)


def pixel_statistic_tokens(img: np.ndarray, feature: str) -> np.ndarray:
    """Reading R14: the feature token [N, FEATURE_DIMS[feature]] of every patch."""
    P = patches(img).astype(np.int64)
    N = P.shape[0]
    one = np.ones((N, 1))
    if feature == "rgb_stats":
        x = P.reshape(N, PATCH * PATCH, 3) / 255.0
        return np.concatenate([x.mean(axis=1), x.std(axis=1), one], axis=1)
    if feature == "color_entropy":
        H = np.zeros((N, 3))
        for c in range(3):
            bins = P[..., c].reshape(N, -1) >> 4
            for i in range(N):
                p = np.bincount(bins[i], minlength=ENTROPY_BINS) / float(PATCH * PATCH)
                p = p[p > 0]
                H[i, c] = float(-(p * np.log2(p)).sum())
        return np.concatenate([H / 4.0, one], axis=1)
    Y = P[..., 0] * LUMA_WEIGHTS[0] + P[..., 1] * LUMA_WEIGHTS[1] + P[..., 2] * LUMA_WEIGHTS[2]   # [N, 14, 14]
    c = Y[:, 1:-1, 1:-1]
    if feature == "edge_density":
        gx = (Y[:, :-2, 2:] + 2 * Y[:, 1:-1, 2:] + Y[:, 2:, 2:]) - (Y[:, :-2, :-2] + 2 * Y[:, 1:-1, :-2] + Y[:, 2:, :-2])
        gy = (Y[:, 2:, :-2] + 2 * Y[:, 2:, 1:-1] + Y[:, 2:, 2:]) - (Y[:, :-2, :-2] + 2 * Y[:, :-2, 1:-1] + Y[:, :-2, 2:])
        thr = int(round(EDGE_TAU * LUMA_SCALE)) ** 2        # exact: magnitudes compared in integers
        e = ((gx * gx + gy * gy) > thr).reshape(N, -1).mean(axis=1)
        return np.stack([e, np.ones(N)], axis=1)
    if feature == "laplacian":
        lap = Y[:, 1:-1, :-2] + Y[:, 1:-1, 2:] + Y[:, :-2, 1:-1] + Y[:, 2:, 1:-1] - 4 * c
        s = lap.reshape(N, -1).astype(np.float64).std(axis=1) / LUMA_SCALE
        return np.stack([s, np.ones(N)], axis=1)
    raise ValueError(feature)


def apc_density_pixel(img: np.ndarray, feature: str, alpha: float = ALPHA, gamma: float = GAMMA,
                      tail_frac: float = TAIL_FRAC, r_min: float = 0.0, r_max: float = 1.0):
    """APC (Eq. 1-6, r, target size) with a pixel-statistic preview in place of T_v (R14)."""
    st = apc_density_tokens(pixel_statistic_tokens(img, feature), alpha, gamma, tail_frac)
    st["r"] = retention_ratio(st["rho"], r_min, r_max)
    st["H_out"], st["W_out"] = target_size(img.shape[0], img.shape[1], st["r"])
    return st


def cubic(t: np.ndarray, a: float = -0.5) -> np.ndarray:
    """Keys' cubic convolution kernel with a = -0.5 (the bicubic of App. B.3)."""
    t = np.abs(t)
    w = np.zeros_like(t)
    m1 = t < 1.0
    m2 = (t >= 1.0) & (t < 2.0)
    w[m1] = ((a + 2.0) * t[m1] - (a + 3.0)) * t[m1] ** 2 + 1.0
    w[m2] = ((a * t[m2] - 5.0 * a) * t[m2] + 8.0 * a) * t[m2] - 4.0 * a
    return w


def resample_matrix(n_in: int, n_out: int) -> np.ndarray:
    """Reading R5: dense [n_out, n_in] matrix of the 1-D antialiased cubic resample."""
    scale = n_in / n_out
    fs = max(scale, 1.0)
    centre = (np.arange(n_out, dtype=np.float64) + 0.5) * scale
    x = np.arange(n_in, dtype=np.float64) + 0.5
    Wm = cubic((x[None, :] - centre[:, None]) / fs)
    return Wm / Wm.sum(axis=1, keepdims=True)


def resample_float(img: np.ndarray, H_out: int, W_out: int) -> np.ndarray:
    """Separable resample of a uint8 HxWx3 image to H_out x W_out, fp64, before rounding."""
    H, W, C = img.shape
    Wy = resample_matrix(H, H_out)
    Wx = resample_matrix(W, W_out)
    x = img.astype(np.float64)
    return np.stack([Wy @ x[:, :, ch] @ Wx.T for ch in range(C)], axis=2)


def apc_resample(img: np.ndarray, H_out: int, W_out: int) -> np.ndarray:
    """App. B.3 bicubic resize to the target size; uint8 out, round half to even."""
    return np.clip(np.rint(resample_float(img, H_out, W_out)), 0, 255).astype(np.uint8)


# ==============================================================================================
# Extract: Dynamic Dual-Attention Extractor (Sec. 3.3)
# ==============================================================================================
def received_attention(q: np.ndarray, k: np.ndarray, scale: float, rows_per_block: int = 512) -> np.ndarray:
    """Column sums of the row-softmax attention matrix of one head.

    q [Nq, d], k [Nk, d] -> a [Nk], a_j = sum_i softmax_j(scale * q_i . k_j).
    Rows are independent, so they are taken a block at a time.
    """
    a = np.zeros(k.shape[0])
    for i0 in range(0, q.shape[0], rows_per_block):
        s = (q[i0:i0 + rows_per_block] @ k.T) * scale
        s -= s.max(axis=1, keepdims=True)
        p = np.exp(s)
        p /= p.sum(axis=1, keepdims=True)
        a += p.sum(axis=0)
    return a


def vit_attn_importance(Q: np.ndarray, K: np.ndarray, cu_seqlens: Sequence[int], scale: float,
                        merge: int = 4) -> np.ndarray:
    """Reading R6 of S_vis (Sec. 3.3; App. B.3: the final ViT block).

    Q, K float64 [sum N, H, d]; images are the row ranges of cu_seqlens.
    Returns S_vis_raw [sum N / merge].
    """
    out: List[np.ndarray] = []
    for b in range(len(cu_seqlens) - 1):
        s0, s1 = int(cu_seqlens[b]), int(cu_seqlens[b + 1])
        a = np.zeros(s1 - s0)
        for h in range(Q.shape[1]):
            a += received_attention(Q[s0:s1, h], K[s0:s1, h], scale)
        out.append(a.reshape(-1, merge).sum(axis=1))
    return np.concatenate(out) if out else np.zeros(0)


def llm_text_visual_importance(Q: np.ndarray, K: np.ndarray, cu_q: Sequence[int], cu_k: Sequence[int],
                               scale: float) -> np.ndarray:
    """Reading R7 of S_llm (Sec. 3.3; App. B.3: layer L_ext = 2).

    Q float64 [sum Tq, Hq, d], K float64 [sum Nv, Hkv, d].  Returns S_llm_raw [sum Nv].
    """
    Hq, Hkv = Q.shape[1], K.shape[1]
    group = Hq // Hkv
    out: List[np.ndarray] = []
    for b in range(len(cu_q) - 1):
        q0, q1 = int(cu_q[b]), int(cu_q[b + 1])
        k0, k1 = int(cu_k[b]), int(cu_k[b + 1])
        u = np.zeros(k1 - k0)
        for h in range(Hq):
            u += received_attention(Q[q0:q1, h], K[k0:k1, h // group], scale)
        out.append(u)
    return np.concatenate(out) if out else np.zeros(0)


# Query sets of the full-sequence S_llm (App. "Impact of Attention Token Sources"): all sequence
# tokens (Vision + Text, the paper's default, App. B.3 "averaged uniformly across all valid
# tokens"), the text tokens only, or the last token only.
QUERY_SETS = ("vision_text", "text", "last")


def query_start(n_seq: int, vis_start: int, n_vis: int, query_set: str) -> int:
    """First query position; the query set is positions query_start .. n_seq - 1.  Positions
    before the visual span cannot attend to it (causal mask), so they are left out."""
    if query_set == "vision_text":
        return vis_start
    if query_set == "text":
        return vis_start + n_vis
    if query_set == "last":
        return n_seq - 1
    raise ValueError(query_set)


def llm_sequence_importance(Q: np.ndarray, K: np.ndarray, cu_seq: Sequence[int], vis_start: Sequence[int],
                            n_vis: Sequence[int], scale: float, query_set: str = "vision_text",
                            rows_per_block: int = 256) -> np.ndarray:
    """Full-sequence S_llm (Sec. 3.3; App. B.3; App. "Impact of Attention Token Sources").

    Q float64 [sum S, Hq, d], K float64 [sum S, Hkv, d]: queries and keys of every position of
    each causal LLM sequence at the extraction layer.  For sequence b with its visual tokens at
    positions v .. v + N_vis - 1 and query set P: S_llm[j] = sum_h sum_{q in P}
    softmax_{k <= q}(scale q_q . k_k)[v + j], the softmax over every earlier position (system,
    visual and text tokens).  GQA head h reads KV head h // (Hq / Hkv).  Returns [sum N_vis].
    """
    Hq, Hkv = Q.shape[1], K.shape[1]
    group = Hq // Hkv
    out: List[np.ndarray] = []
    for b in range(len(cu_seq) - 1):
        s0, s1 = int(cu_seq[b]), int(cu_seq[b + 1])
        S, v, nv = s1 - s0, int(vis_start[b]), int(n_vis[b])
        q_lo = query_start(S, v, nv, query_set)
        u = np.zeros(nv)
        for h in range(Hq):
            Kh = K[s0:s1, h // group]
            for i0 in range(q_lo, S, rows_per_block):
                i1 = min(S, i0 + rows_per_block)
                logits = (Q[s0 + i0:s0 + i1, h] @ Kh.T) * scale           # [rows, S]
                pos_q = np.arange(i0, i1)[:, None]
                logits = np.where(np.arange(S)[None, :] <= pos_q, logits, -np.inf)   # causal
                logits -= logits.max(axis=1, keepdims=True)
                p = np.exp(logits)
                p /= p.sum(axis=1, keepdims=True)
                u += p[:, v:v + nv].sum(axis=0)
        out.append(u)
    return np.concatenate(out) if out else np.zeros(0)


def min_max(x: np.ndarray) -> np.ndarray:
    """Sec. 3.3: min-max normalisation to [0, 1]; a constant map becomes 0 (R8)."""
    lo, hi = float(x.min()), float(x.max())
    if hi == lo:
        return np.zeros_like(x, dtype=np.float64)
    return (x - lo) / (hi - lo)


# Fusion modes: Eq. 7, and the fusion ablations of Sec. 4 "Effect of Attention Fusion in DDAE"
# (Only LLM-Attn, Only ViT-Attn, Fixed Fusion with 0.5 on each signal).
FUSION_WEIGHTS = {"only_llm": (1.0, 0.0), "only_vit": (0.0, 1.0), "fixed": (0.5, 0.5)}


def ddae_fuse(s_llm_raw: np.ndarray, s_vis_raw: np.ndarray, tau: float = TAU,
              fusion: str = "adaptive") -> Dict[str, object]:
    """Eq. 7 and S_final = alpha_w * S_llm + beta_w * S_vis for one image."""
    S_llm = min_max(np.asarray(s_llm_raw, dtype=np.float64))
    S_vis = min_max(np.asarray(s_vis_raw, dtype=np.float64))
    sigma_llm = float(S_llm.std())      # population deviation (R8)
    sigma_vis = float(S_vis.std())
    if fusion == "adaptive":
        z = np.array([sigma_llm, sigma_vis]) / tau
        e = np.exp(z - z.max())
        w = e / e.sum()
    else:
        w = np.array(FUSION_WEIGHTS[fusion])
    S_final = w[0] * S_llm + w[1] * S_vis
    return dict(S_llm=S_llm, S_vis=S_vis, sigma_llm=sigma_llm, sigma_vis=sigma_vis,
                alpha_w=float(w[0]), beta_w=float(w[1]), S_final=S_final)


def budget(n_vis: int, frac: float) -> int:
    """Reading R9: K = floor(frac * N_vis + 0.5) clamped to [0, N_vis]."""
    return int(min(max(math.floor(frac * n_vis + 0.5), 0), n_vis))


def top_k_ascending(S_final: np.ndarray, K: int) -> np.ndarray:
    """Sec. 3.3: indices of the K highest S_final (ties: lower index), in ascending order."""
    n = len(S_final)
    order = np.lexsort((np.arange(n), -np.asarray(S_final, dtype=np.float64)))
    return np.sort(order[:K]).astype(np.int64)


def ddae_select(s_llm_raw: np.ndarray, s_vis_raw: np.ndarray, cu_v: Sequence[int],
                keep: Sequence[int], tau: float = TAU, fusion: str = "adaptive") -> Dict[str, np.ndarray]:
    """Per image: fuse, then keep the top K_b tokens.  Kept rows are global (cu_v-offset) indices."""
    S_final, weights, kept = [], [], []
    for b in range(len(cu_v) - 1):
        v0, v1 = int(cu_v[b]), int(cu_v[b + 1])
        f = ddae_fuse(s_llm_raw[v0:v1], s_vis_raw[v0:v1], tau, fusion)
        S_final.append(f["S_final"])
        weights.append([f["alpha_w"], f["beta_w"]])
        kept.append(top_k_ascending(f["S_final"], int(keep[b])) + v0)
    return dict(S_final=np.concatenate(S_final), weights=np.asarray(weights),
                kept=np.concatenate(kept) if kept else np.zeros(0, dtype=np.int64))


def gather_rows(E: np.ndarray, idx: np.ndarray) -> np.ndarray:
    """Sec. 3.3: the kept visual rows form the pruned LLM context."""
    return E[np.asarray(idx, dtype=np.int64)]


def budget_vanilla(n_vis_vanilla: int, n_vis_condensed: int, frac: float) -> int:
    """App. C: the final ratio B = p1 p2 is relative to Vanilla, so K = round(B * N_vis_vanilla)
    (reading R9's rounding), capped at the tokens left after condensation."""
    return min(budget(n_vis_vanilla, frac), max(n_vis_condensed, 0))


def prune_rows(n_pre: int, vis_start: int, n_vis: int, kept_local: Sequence[int]) -> np.ndarray:
    """Sec. 3.3 / App. C: rows of the pruned LLM sequence, S_post = T + N_keep positions: every
    position outside the visual span, and the kept visual positions, in sequence order."""
    keep = np.ones(n_pre, dtype=bool)
    keep[vis_start:vis_start + n_vis] = False
    keep[vis_start + np.asarray(kept_local, dtype=np.int64)] = True
    return np.nonzero(keep)[0]
