"""Pins of the fp64 oracle against things other than itself.

Each test checks the oracle against a hand-derived closed form (tests/golden),
a brute-force pure-Python evaluation on tiny inputs, an independent library
routine, or an invariant that the mathematics fixes.  No GPU is needed.
"""
import math

import numpy as np
import pytest
import torch

from oracle import pace_oracle as O
from paper_2608_27206_gb300 import synth


# ----------------------------------------------------------------------------------------------
# Hyper-parameters
# ----------------------------------------------------------------------------------------------
def test_hyperparameters_match_paper(golden):
    g = golden("paper_hyperparameters.txt")
    assert O.ALPHA == g["alpha"] and O.GAMMA == g["gamma"] and O.TAU == g["tau"]
    assert O.TAIL_FRAC == g["tail_frac"]
    assert O.MERGE_UNIT == g["merge_unit"] and O.PATCH == g["patch"]


# ----------------------------------------------------------------------------------------------
# APC density (Eq. 1-6)
# ----------------------------------------------------------------------------------------------
def test_two_orthogonal_tokens_closed_form(golden):
    g = golden("apc_two_orthogonal_tokens.txt")
    T = np.array([[3.0, 0.0, 0.0], [0.0, 0.5, 0.0]])   # orthogonal, unequal norms
    st = O.apc_density_tokens(T)
    assert st["k_tail"] == g["k_tail"]
    for key in ("phi", "rho_g", "d_top", "rho_d", "rho"):
        assert st[key] == pytest.approx(g[key], abs=1e-14), key
    np.testing.assert_allclose(st["d"], [g["d"], g["d"]], atol=1e-14)


def _phi_brute(T):
    """Pure-Python double loop over all pairs (Eq. 1 written out)."""
    N = len(T)
    tot = 0.0
    for i in range(N):
        for j in range(N):
            dot = sum(a * b for a, b in zip(T[i], T[j]))
            ni = math.sqrt(sum(a * a for a in T[i]))
            nj = math.sqrt(sum(b * b for b in T[j]))
            tot += dot / (ni * nj)
    return tot / (N * N)


def _density_brute(T, alpha=0.6, gamma=1.5, tail=0.1):
    N, D = len(T), len(T[0])
    norms = [math.sqrt(sum(a * a for a in t)) for t in T]
    Tn = [[a / n for a in t] for t, n in zip(T, norms)]
    c = [sum(Tn[i][k] for i in range(N)) / N for k in range(D)]
    cn = math.sqrt(sum(a * a for a in c))
    ch = [a / cn for a in c]
    d = [math.sqrt(sum((Tn[i][k] - ch[k]) ** 2 for k in range(D))) for i in range(N)]
    kt = max(1, int(tail * N + 0.5))
    top = sorted(d, reverse=True)[:kt]
    d_top = sum(top) / kt
    phi = _phi_brute(T)
    rho_d = min(d_top / gamma, 1.0)
    return dict(phi=phi, d=d, k_tail=kt, d_top=d_top, rho_d=rho_d,
                rho=alpha * (1 - phi) + (1 - alpha) * rho_d)


@pytest.mark.parametrize("N,D,seed", [(1, 4, 0), (3, 5, 1), (7, 3, 2), (23, 6, 3), (40, 9, 4)])
def test_density_brute_force(N, D, seed):
    rng = np.random.default_rng(seed)
    T = rng.standard_normal((N, D)) + 0.3
    st = O.apc_density_tokens(T)
    bf = _density_brute(T.tolist())
    assert st["phi"] == pytest.approx(bf["phi"], rel=1e-12, abs=1e-14)
    assert st["k_tail"] == bf["k_tail"]
    np.testing.assert_allclose(st["d"], bf["d"], rtol=1e-12, atol=1e-14)
    for key in ("d_top", "rho_d", "rho"):
        assert st[key] == pytest.approx(bf[key], rel=1e-12, abs=1e-14), key


def test_phi_equals_squared_norm_of_mean():
    """Identity: (1/N^2) sum_ij cos_ij = |mean of unit tokens|^2."""
    rng = np.random.default_rng(5)
    T = rng.uniform(0, 1, (300, 589))
    st = O.apc_density_tokens(T)
    assert st["phi"] == pytest.approx(float(st["c"] @ st["c"]), rel=1e-12)


def test_patch_tokens_layout():
    """Patch i of the raster grid holds the 14x14x3 pixels of that cell, then the constant 1."""
    rng = np.random.default_rng(6)
    img = rng.integers(0, 256, (28, 42, 3), dtype=np.uint8)
    T = O.patch_tokens(img)
    assert T.shape == (6, 589)
    for py in range(2):
        for px in range(3):
            cell = img[py * 14:(py + 1) * 14, px * 14:(px + 1) * 14].astype(np.float64) / 255.0
            np.testing.assert_array_equal(T[py * 3 + px, :588], cell.reshape(-1))
    np.testing.assert_array_equal(T[:, 588], 1.0)


def test_constant_image_minimal_density():
    """A constant image: all tokens equal -> phi = 1, d = 0, rho = 0, smallest target."""
    for v in (0, 17, 255):
        img = np.full((112, 168, 3), v, dtype=np.uint8)
        st = O.apc_density(img)
        assert abs(st["phi"] - 1.0) < 1e-12
        assert np.abs(st["d"]).max() < 1e-7
        assert abs(st["rho"]) < 1e-7
        assert (st["H_out"], st["W_out"]) == (28, 28)


def test_redundancy_and_detail_properties():
    """Sec. 3.2: more uniform area -> lower rho_g; sparse detail on a flat page -> higher rho_d."""
    rng = np.random.default_rng(7)
    H = W = 224
    rhos = []
    noise = rng.integers(0, 256, (H, W, 3), dtype=np.uint8)
    for n_noisy in (0, 2, 6, 16):                 # 4x4 tiles of 56 px; the rest flat grey
        img = np.full((H, W, 3), 128, dtype=np.uint8)
        for t in range(n_noisy):
            y, x = (t // 4) * 56, (t % 4) * 56
            img[y:y + 56, x:x + 56] = noise[y:y + 56, x:x + 56]
        rhos.append(O.apc_density(img)["rho_g"])
    assert all(a < b for a, b in zip(rhos, rhos[1:])), rhos
    flat = np.full((H, W, 3), 240, dtype=np.uint8)
    detail = flat.copy()
    cells = rng.permutation((H // 14) * (W // 14))[:30]          # ~12 % of the patches: dark marks
    for c in cells:
        y, x = (c // (W // 14)) * 14, (c % (W // 14)) * 14
        detail[y:y + 14, x:x + 14] = rng.integers(0, 60, (14, 14, 3))
    a, b = O.apc_density(flat), O.apc_density(detail)
    assert a["rho_d"] < 1e-7 and b["rho_d"] > 0.3
    assert b["rho_g"] < 0.1 < b["rho_d"]          # globally redundant, locally detailed


def test_retention_and_target_size():
    assert O.retention_ratio(0.3) == 0.3
    assert O.retention_ratio(-0.01) == 0.0
    assert O.retention_ratio(0.8, r_max=0.5) == 0.5      # hard budget cap
    assert O.target_size(2156, 3836, 1.0) == (2156, 3836)
    assert O.target_size(2156, 3836, 0.25) == (1092, 1932)   # 38.5 -> 39 and 68.5 -> 69 units (half up)
    assert O.target_size(448, 448, 0.0) == (28, 28)
    assert O.target_size(448, 448, 0.5) == (308, 308)        # 316.8 / 28 = 11.31 -> 11


# ----------------------------------------------------------------------------------------------
# Bicubic resample
# ----------------------------------------------------------------------------------------------
@pytest.mark.parametrize("shape_in,shape_out", [((56, 84), (28, 28)), ((56, 84), (56, 84)),
                                                ((98, 70), (42, 56)), ((140, 140), (28, 70)),
                                                ((84, 56), (37, 19)), ((224, 308), (112, 140))])
def test_resample_matches_torch_antialiased_bicubic(shape_in, shape_out):
    """Independent library routine: torch's antialiased bicubic (a = -0.5) in float64."""
    rng = np.random.default_rng(8)
    img = rng.integers(0, 256, shape_in + (3,), dtype=np.uint8)
    ref = O.resample_float(img, *shape_out)
    t = torch.from_numpy(img.astype(np.float64)).permute(2, 0, 1)[None]
    tt = torch.nn.functional.interpolate(t, size=shape_out, mode="bicubic", antialias=True,
                                         align_corners=False)[0].permute(1, 2, 0).numpy()
    np.testing.assert_allclose(ref, tt, atol=1e-9)


def test_resample_invariants():
    rng = np.random.default_rng(9)
    img = rng.integers(0, 256, (84, 112, 3), dtype=np.uint8)
    np.testing.assert_array_equal(O.apc_resample(img, 84, 112), img)          # r = 1: identity
    const = np.full((84, 112, 3), 201, dtype=np.uint8)
    for ho, wo in ((28, 28), (56, 84), (42, 28)):
        np.testing.assert_array_equal(O.apc_resample(const, ho, wo), 201)     # constant stays
    ramp = np.tile(np.arange(112, dtype=np.uint8)[None, :, None] * 2, (84, 1, 3))
    out = O.resample_float(ramp, 42, 56)                                        # 2x down
    # interior of a linear ramp stays linear: x_out = 2 * (2 o + 0.5)
    np.testing.assert_allclose(out[:, 2:-2, 0], np.tile(4 * np.arange(56)[2:-2] + 1.0, (42, 1)), atol=1e-9)


def test_cubic_kernel_values():
    t = np.array([0.0, 0.5, 1.0, 1.5, 2.0, 2.5])
    # Keys (1981), a = -0.5: W(0)=1, W(0.5)=0.5625, W(1)=0, W(1.5)=-0.0625, W(>=2)=0
    np.testing.assert_allclose(O.cubic(t), [1.0, 0.5625, 0.0, -0.0625, 0.0, 0.0], atol=1e-15)


# ----------------------------------------------------------------------------------------------
# Attention importance
# ----------------------------------------------------------------------------------------------
def _received_brute(q, k, scale):
    Nq, Nk = len(q), len(k)
    a = [0.0] * Nk
    for i in range(Nq):
        s = [scale * sum(x * y for x, y in zip(q[i], k[j])) for j in range(Nk)]
        m = max(s)
        e = [math.exp(v - m) for v in s]
        z = sum(e)
        for j in range(Nk):
            a[j] += e[j] / z
    return a


def test_vit_importance_brute_force():
    rng = np.random.default_rng(10)
    cu = [0, 8, 20]
    Q = rng.standard_normal((20, 2, 5)) * 1.5
    K = rng.standard_normal((20, 2, 5))
    out = O.vit_attn_importance(Q, K, cu, 0.7, merge=4)
    ref = []
    for b in range(2):
        a = np.zeros(cu[b + 1] - cu[b])
        for h in range(2):
            a += _received_brute(Q[cu[b]:cu[b + 1], h].tolist(), K[cu[b]:cu[b + 1], h].tolist(), 0.7)
        ref.append(a.reshape(-1, 4).sum(1))
    np.testing.assert_allclose(out, np.concatenate(ref), rtol=1e-12)


def test_vit_importance_torch_softmax_and_invariants():
    rng = np.random.default_rng(11)
    N, H, d = 64, 3, 16
    Q = rng.standard_normal((N, H, d))
    K = rng.standard_normal((N, H, d))
    out = O.vit_attn_importance(Q, K, [0, N], 1 / math.sqrt(d), merge=1)
    qt, kt = torch.from_numpy(Q), torch.from_numpy(K)
    P = torch.softmax(torch.einsum("ihd,jhd->hij", qt, kt) / math.sqrt(d), dim=-1)
    np.testing.assert_allclose(out, P.sum(dim=(0, 1)).numpy(), rtol=1e-12)
    assert out.sum() == pytest.approx(N * H, rel=1e-13)          # rows sum to 1
    Kc = np.repeat(K[:1], N, axis=0)                              # all keys equal
    np.testing.assert_allclose(O.vit_attn_importance(Q, Kc, [0, N], 0.3, merge=4), 4 * H, rtol=1e-13)


def test_llm_importance_gqa_equals_repeated_kv_mha():
    """GQA with G query heads per KV head == MHA on K repeated G times per head."""
    rng = np.random.default_rng(12)
    Hq, Hkv, d = 6, 2, 8
    cu_q, cu_k = [0, 5, 12], [0, 9, 13]
    Q = rng.standard_normal((12, Hq, d))
    K = rng.standard_normal((13, Hkv, d))
    out = O.llm_text_visual_importance(Q, K, cu_q, cu_k, 0.4)
    Krep = np.repeat(K, Hq // Hkv, axis=1)        # head h <- KV head h // 3
    ref = []
    for b in range(2):
        u = np.zeros(cu_k[b + 1] - cu_k[b])
        for h in range(Hq):
            u += _received_brute(Q[cu_q[b]:cu_q[b + 1], h].tolist(),
                                 Krep[cu_k[b]:cu_k[b + 1], h].tolist(), 0.4)
        ref.append(u)
    np.testing.assert_allclose(out, np.concatenate(ref), rtol=1e-12)
    assert out[:9].sum() == pytest.approx(5 * Hq, rel=1e-13)
    assert out[9:].sum() == pytest.approx(7 * Hq, rel=1e-13)


# ----------------------------------------------------------------------------------------------
# DDAE fusion, budget, top-K, gather
# ----------------------------------------------------------------------------------------------
def test_ddae_four_token_closed_form(golden):
    g = golden("ddae_four_tokens.txt")
    f = O.ddae_fuse(np.array(g["s_llm_raw"]), np.array(g["s_vis_raw"]))
    assert f["sigma_llm"] == pytest.approx(g["sigma_llm"], abs=1e-15)
    assert f["sigma_vis"] == pytest.approx(g["sigma_vis"], abs=1e-15)
    assert f["alpha_w"] == pytest.approx(g["alpha_w"], abs=1e-15)
    assert f["beta_w"] == pytest.approx(g["beta_w"], abs=1e-15)
    np.testing.assert_allclose(f["S_final"], g["s_final"], atol=1e-15)
    assert O.top_k_ascending(f["S_final"], 2).tolist() == [int(x) for x in g["kept_top2"]]
    assert O.top_k_ascending(f["S_final"], 1).tolist() == [int(g["kept_top1"])]


def test_ddae_limits():
    rng = np.random.default_rng(13)
    x = rng.uniform(size=50)
    f = O.ddae_fuse(x, 3 * x + 1)         # same normalised map -> equal sigma -> 0.5 / 0.5
    assert f["alpha_w"] == pytest.approx(0.5, abs=1e-15) and f["beta_w"] == pytest.approx(0.5, abs=1e-15)
    np.testing.assert_allclose(f["S_final"], (x - x.min()) / (x.max() - x.min()), atol=1e-15)
    f = O.ddae_fuse(np.full(7, 2.0), rng.uniform(size=7))
    assert np.all(f["S_llm"] == 0) and f["sigma_llm"] == 0.0
    assert f["alpha_w"] + f["beta_w"] == pytest.approx(1.0, abs=1e-15)
    assert f["beta_w"] > 0.5               # the sharper map gets the larger weight


def test_budgets(golden):
    g = golden("workload_budgets.txt")
    for key in ("img448", "img1344", "frame1904"):
        n, p, k = g[key]
        assert O.budget(int(n), p) == int(k)
    assert synth.make_workload("img4k", parts=()).n_patches == [int(g["patches_4k"][2])]
    assert synth.make_workload("img4k", parts=()).n_vis == [int(g["tokens_4k"][2])]
    assert O.budget(10, 0.0) == 0 and O.budget(10, 1.0) == 10 and O.budget(10, 2.0) == 10
    assert O.budget(10549, 0.05) == 527 and O.budget(10549, 0.10) == 1055


@pytest.mark.parametrize("seed", range(5))
def test_top_k_against_full_sort(seed):
    rng = np.random.default_rng(seed)
    n = int(rng.integers(1, 200))
    s = np.round(rng.uniform(size=n), 1)         # many ties
    for K in (0, 1, n // 3, n):
        ranked = sorted(range(n), key=lambda i: (-s[i], i))
        assert O.top_k_ascending(s, K).tolist() == sorted(ranked[:K])


def test_ddae_select_ragged_offsets():
    rng = np.random.default_rng(14)
    cu = [0, 5, 5 + 9, 5 + 9 + 4]
    sl, sv = rng.uniform(size=18), rng.uniform(size=18)
    res = O.ddae_select(sl, sv, cu, [2, 0, 4])
    assert len(res["kept"]) == 6
    assert res["kept"][:2].min() >= 0 and res["kept"][:2].max() < 5
    assert res["kept"][2:].tolist() == [14, 15, 16, 17]
    np.testing.assert_allclose(res["weights"].sum(1), 1.0, atol=1e-15)


def test_gather_rows():
    E = np.arange(40, dtype=np.uint16).reshape(10, 4)
    np.testing.assert_array_equal(O.gather_rows(E, [3, 0, 9]), E[[3, 0, 9]])


def test_ddae_fusion_ablation_modes():
    """Fusion ablations (Sec. 4): with one weight at 1 the kept set is the top of that map alone
    (checked against a plain sort of the single map); fixed fusion is the mean of the two maps
    and equals Eq. 7 when the two deviations are equal."""
    rng = np.random.default_rng(12)
    sl, sv = rng.gamma(0.5, 2.0, 500), rng.lognormal(0, 1, 500)
    for mode, raw in (("only_llm", sl), ("only_vit", sv)):
        f = O.ddae_fuse(sl, sv, fusion=mode)
        z = (raw - raw.min()) / (raw.max() - raw.min())
        np.testing.assert_allclose(f["S_final"], z, rtol=0, atol=1e-15)
        K = 37
        brute = np.sort(sorted(range(500), key=lambda i: (-z[i], i))[:K])
        np.testing.assert_array_equal(O.top_k_ascending(f["S_final"], K), brute)
    f = O.ddae_fuse(sl, sv, fusion="fixed")
    assert (f["alpha_w"], f["beta_w"]) == (0.5, 0.5)
    np.testing.assert_allclose(f["S_final"], 0.5 * (f["S_llm"] + f["S_vis"]), atol=1e-15)
    a = rng.normal(size=64)
    g_adapt = O.ddae_fuse(a, -a)                       # mirrored maps: equal deviations
    g_fixed = O.ddae_fuse(a, -a, fusion="fixed")
    np.testing.assert_allclose(g_adapt["S_final"], g_fixed["S_final"], atol=1e-12)


def test_preview_tokens_zero_rows_and_identity():
    """Reading R10 on preview tokens: zero rows are t_hat = 0; Eq. 1 (literal double sum) still
    equals |c|^2; with every token equal, phi = 1, rho_g = 0, all d_i = 0."""
    rng = np.random.default_rng(21)
    T = rng.normal(size=(40, 24))
    T[[3, 17]] = 0.0
    st = O.apc_density_tokens(T)
    Tn = [t / np.linalg.norm(t) if np.linalg.norm(t) > 0 else np.zeros_like(t) for t in T]
    brute = sum(float(a @ b_) for a in Tn for b_ in Tn) / (40 * 40)
    assert st["phi"] == pytest.approx(brute, rel=1e-12)
    assert st["phi"] == pytest.approx(float(st["c"] @ st["c"]), rel=1e-12)
    assert st["d"][3] == pytest.approx(1.0) and st["d"][17] == pytest.approx(1.0)   # |0 - c_hat| = 1
    same = np.tile(rng.normal(size=(1, 24)), (30, 1))
    st2 = O.apc_density_preview(same, 280, 420)
    assert st2["phi"] == pytest.approx(1.0) and st2["rho_g"] == pytest.approx(0.0, abs=1e-12)
    assert np.all(np.abs(st2["d"]) < 1e-7)
    assert (st2["H_out"], st2["W_out"]) == (28, 28)                                # r = 0


def test_prune_rows_against_position_loop():
    """The pruned sequence keeps text positions and the kept visual positions, in order
    (checked against a plain loop over positions)."""
    rng = np.random.default_rng(3)
    for _ in range(50):
        n_vis = int(rng.integers(0, 60))
        pre, post = int(rng.integers(0, 20)), int(rng.integers(0, 20))
        kept = np.sort(rng.choice(n_vis, size=int(rng.integers(0, n_vis + 1)), replace=False)) if n_vis else []
        rows = O.prune_rows(pre + n_vis + post, pre, n_vis, kept)
        ks = set(int(k) for k in kept)
        expect = [p for p in range(pre + n_vis + post) if not (pre <= p < pre + n_vis) or (p - pre) in ks]
        np.testing.assert_array_equal(rows, expect)
        assert len(rows) == pre + post + len(kept)       # S_post = T + N_keep


def test_llm_sequence_importance_brute_force_and_mass():
    """Full-sequence S_llm: a materialised causal softmax written as plain loops (tiny sizes),
    and the attention mass: each query's softmax sums to 1 over its keys, so the visual mass is
    at most |P| * Hq, with equality when the visual span is the whole prefix of every query."""
    rng = np.random.default_rng(8)
    S, v, nv, Hq, Hkv, d = 23, 5, 9, 4, 2, 6
    Q = rng.normal(size=(S, Hq, d))
    K = rng.normal(size=(S, Hkv, d))
    scale = 0.4
    for qs in O.QUERY_SETS:
        got = O.llm_sequence_importance(Q, K, [0, S], [v], [nv], scale, qs)
        q_lo = {"vision_text": v, "text": v + nv, "last": S - 1}[qs]
        want = np.zeros(nv)
        for h in range(Hq):
            for q in range(q_lo, S):
                w = [math.exp(scale * float(Q[q, h] @ K[k, h // 2])) for k in range(q + 1)]
                z = sum(w)
                for j in range(nv):
                    if v + j <= q:
                        want[j] += w[v + j] / z
        np.testing.assert_allclose(got, want, rtol=1e-12, atol=1e-15)
        assert got.sum() <= (S - q_lo) * Hq + 1e-9
    # image at the start of the sequence, text queries only, keys = visual + earlier text:
    # with text keys scored -inf-like (huge negative), all mass goes to the visual keys
    K2 = K.copy()
    K2[nv:] = 0.0
    Q2 = Q.copy()
    got = O.llm_sequence_importance(Q2 * 0 + 1.0, K2 * 0 + np.r_[np.ones(nv), np.zeros(S - nv)][:, None, None],
                                    [0, S], [0], [nv], 50.0, "text")
    assert got.sum() == pytest.approx((S - nv) * Hq, rel=1e-9)


# ----------------------------------------------------------------------------------------------
# Pixel-statistic preview features (App. "Shallow Feature Preview Ablation"; reading R14)
# ----------------------------------------------------------------------------------------------
def _one_patch(pix):
    """A 14 x 14 image of one patch from a 14 x 14 grey-level array (R = G = B)."""
    return np.repeat(np.asarray(pix, dtype=np.uint8)[:, :, None], 3, axis=2)


def test_pixel_features_two_tone_closed_forms():
    # left 7 columns black, right 7 white: every channel is 0 or 1 with probability 1/2, so
    # mean = std = 1/2; two of 16 bins hold half the pixels each: 1 bit -> 1/4 after scaling.
    # Sobel: only interior columns 6 and 7 straddle the boundary (2 x 12 of 144 pixels), with
    # |G| = 4 (one full step weighted 1 + 2 + 1) > 0.25.  Laplacian: +1 on column 6 (one white
    # neighbour), -1 on column 7 (one black neighbour), 0 elsewhere: std = sqrt(24 / 144).
    pix = np.zeros((14, 14))
    pix[:, 7:] = 255
    img = _one_patch(pix)
    np.testing.assert_allclose(O.pixel_statistic_tokens(img, "rgb_stats")[0], [0.5] * 6 + [1.0], atol=1e-15)
    np.testing.assert_allclose(O.pixel_statistic_tokens(img, "color_entropy")[0], [0.25] * 3 + [1.0], atol=1e-15)
    np.testing.assert_allclose(O.pixel_statistic_tokens(img, "edge_density")[0], [1 / 6, 1.0], atol=1e-15)
    np.testing.assert_allclose(O.pixel_statistic_tokens(img, "laplacian")[0], [math.sqrt(1 / 6), 1.0], atol=1e-15)
    # the same split across rows exercises the other gradient and neighbour directions
    imgT = _one_patch(pix.T)
    np.testing.assert_allclose(O.pixel_statistic_tokens(imgT, "edge_density")[0], [1 / 6, 1.0], atol=1e-15)
    np.testing.assert_allclose(O.pixel_statistic_tokens(imgT, "laplacian")[0], [math.sqrt(1 / 6), 1.0], atol=1e-15)


def test_pixel_features_checkerboard_and_ramp():
    # 1-pixel checkerboard: the columns on either side of a pixel carry the same colours, so both
    # Sobel components vanish (edge density 0), while every Laplacian is +-4 (all four neighbours
    # opposite): std 4.  A ramp of one grey level per column has zero Laplacian and a Sobel
    # magnitude of 4 * 2 / 255 < 0.25.
    y, x = np.mgrid[0:14, 0:14]
    img = _one_patch(((x + y) % 2) * 255)
    assert O.pixel_statistic_tokens(img, "edge_density")[0, 0] == 0.0
    np.testing.assert_allclose(O.pixel_statistic_tokens(img, "laplacian")[0], [4.0, 1.0], atol=1e-12)
    np.testing.assert_allclose(O.pixel_statistic_tokens(img, "color_entropy")[0, :3], [0.25] * 3, atol=1e-15)
    ramp = _one_patch(np.tile(np.arange(14) + 40, (14, 1)))
    assert O.pixel_statistic_tokens(ramp, "laplacian")[0, 0] == 0.0
    assert O.pixel_statistic_tokens(ramp, "edge_density")[0, 0] == 0.0


def test_pixel_features_invariants_and_density():
    rng = np.random.default_rng(21)
    img = rng.integers(0, 256, size=(42, 56, 3), dtype=np.uint8)
    for f in O.PIXEL_FEATURES:
        T = O.pixel_statistic_tokens(img, f)
        assert T.shape == (12, O.FEATURE_DIMS[f]) and np.all(T[:, -1] == 1.0)
        # a constant image gives one token for every patch: phi = 1, d = 0
        st = O.apc_density_pixel(np.full((28, 42, 3), 77, np.uint8), f)
        assert abs(st["phi"] - 1.0) < 1e-12 and np.all(np.abs(st["d"]) < 1e-7)
    # the first-order statistics do not depend on where a pixel sits in its patch
    perm = rng.permutation(196)
    P = O.patches(img)[0].reshape(196, 3)[perm].reshape(14, 14, 3)
    for f in ("rgb_stats", "color_entropy"):
        np.testing.assert_allclose(O.pixel_statistic_tokens(P, f)[0], O.pixel_statistic_tokens(img, f)[0], atol=1e-12)
    ent = O.pixel_statistic_tokens(img, "color_entropy")[:, :3]
    assert np.all(ent >= 0) and np.all(ent <= 1.0)
