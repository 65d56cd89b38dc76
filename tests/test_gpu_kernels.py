"""GPU parity of every libpace entry point against the fp64 oracle on small seeded inputs.

Sizes span several 128-row tiles with ragged tails, multi-image batches, and the
degenerate cases (one patch, one token, K = 0 or N, constant maps, ties).
"""
import math

import numpy as np
import pytest
import torch

from oracle import pace_oracle as O
from paper_2608_27206_gb300 import synth
from tests.helpers import assert_distances_close, assert_kept_matches, assert_scores_close, bf16_tensor, f64

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def pace():
    from paper_2608_27206_gb300 import build
    build.build()
    from paper_2608_27206_gb300 import pace as P
    P.pace_init(0)
    P.pace_device_status(clear=True)
    return P


def _no_device_error(P):
    code, where = P.pace_device_status(clear=True)
    assert code == 0, (code, where)


# ----------------------------------------------------------------------------------------------
# gather
# ----------------------------------------------------------------------------------------------
@pytest.mark.parametrize("n_rows,row_elems,n_idx", [(300, 3584, 50), (1, 3584, 3), (97, 8, 200), (64, 5, 7)])
def test_gather_bit_exact(pace, n_rows, row_elems, n_idx):
    rng = np.random.default_rng(n_rows + n_idx)
    E = rng.integers(-32768, 32767, size=(n_rows, row_elems), dtype=np.int16)
    idx = rng.integers(0, n_rows, size=n_idx).astype(np.int32)
    out = pace.pace_gather(torch.from_numpy(E).cuda(), torch.from_numpy(idx).cuda()).cpu().numpy()
    np.testing.assert_array_equal(out, O.gather_rows(E, idx))
    _no_device_error(pace)


def test_gather_empty_and_bad_index(pace):
    E = torch.arange(64 * 16, dtype=torch.int16, device="cuda").view(64, 16)
    assert pace.pace_gather(E, torch.zeros(0, dtype=torch.int32, device="cuda")).numel() == 0
    idx = torch.tensor([3, 64, -1, 5], dtype=torch.int32, device="cuda")   # two out of range
    out = pace.pace_gather(E, idx).cpu().numpy()
    ref = E.cpu().numpy()
    np.testing.assert_array_equal(out[0], ref[3])
    np.testing.assert_array_equal(out[3], ref[5])
    assert not out[1].any() and not out[2].any()
    code, where = pace.pace_device_status(clear=True)
    assert code == pace.PACE_ERR_INVALID_ARG and where == 10


# ----------------------------------------------------------------------------------------------
# APC density + resample
# ----------------------------------------------------------------------------------------------
def _density(pace, images, params=None, **kw):
    buf, off = synth.pack_images(images)
    H = [im.shape[0] for im in images]
    W = [im.shape[1] for im in images]
    d, st = pace.pace_apc_density(torch.from_numpy(buf).cuda(), off, H, W, params=params)
    return d.cpu().numpy(), pace.stats_dict(st)


def _check_density(d, st, images, alpha=0.6, gamma=1.5, tail=0.1, r_min=0.0, r_max=1.0):
    p0 = 0
    for im, s in zip(images, st):
        ref = O.apc_density(im, alpha, gamma, tail, r_min, r_max)
        n = ref["N"]
        assert s["n_patches"] == n and s["k_tail"] == ref["k_tail"]
        # d_i are distances between unit vectors (O(1)); 1e-5 absolute covers fp32 rounding
        # where the exact distance is 0 (identical tokens)
        assert_distances_close(d[p0:p0 + n], ref["d"], what="d_i")
        for k in ("phi", "d_top", "rho_d", "r"):
            assert abs(s[k] - ref[k]) <= 2e-3 * max(abs(ref[k]), 1e-3), (k, s[k], ref[k])
        assert abs(s["rho_g"] - ref["rho_g"]) <= 2e-3 * max(abs(ref["rho_g"]), 1e-3) + 2e-6
        assert abs(s["rho"] - ref["rho"]) <= 2e-3 * max(abs(ref["rho"]), 1e-3) + 2e-6
        # target size: an integer decided in floating point; equal unless the oracle's value
        # sits within the score tolerance of a rounding boundary
        for side, key in ((im.shape[0], "h_out"), (im.shape[1], "w_out")):
            x = side * math.sqrt(max(ref["r"], 0.0)) / 28 + 0.5
            near = abs(x - round(x)) < 2e-3 * x
            exp = ref["H_out"] if key == "h_out" else ref["W_out"]
            assert s[key] == exp or (near and abs(s[key] - exp) == 28), (key, s[key], exp)
        p0 += n


@pytest.mark.parametrize("shape,tiles,hf", [((28, 28), (1, 1), 1.0), ((14, 14), (1, 1), 1.0),
                                             ((112, 154), (2, 2), 0.5), ((448, 448), (4, 4), 0.5),
                                             ((70, 462), (3, 1), 0.3), ((322, 98), (2, 5), 0.6)])
def test_density_single(pace, shape, tiles, hf):
    rng = np.random.default_rng(shape[0] * 7 + shape[1])
    img = synth.make_image(rng, shape[0], shape[1], tiles[0], tiles[1], hf)
    d, st = _density(pace, [img])
    _check_density(d, st, [img])
    _no_device_error(pace)


def test_density_batch_and_params(pace):
    rng = np.random.default_rng(3)
    imgs = [synth.make_image(rng, h, w, 3, 2, f) for h, w, f in
            [(224, 448, 0.2), (56, 56, 0.9), (616, 532, 0.4), (1008, 28, 0.1), (42, 70, 0.5)]]
    d, st = _density(pace, imgs)
    _check_density(d, st, imgs)
    p = pace.apc_params(alpha=0.3, gamma=0.8, tail_frac=0.05, r_min=0.1, r_max=0.4)
    d, st = _density(pace, imgs, params=p)
    _check_density(d, st, imgs, alpha=0.3, gamma=0.8, tail=0.05, r_min=0.1, r_max=0.4)
    # the static-resolution baselines (a fixed ratio for every image): r_min = r_max = 0.5
    p = pace.apc_params(r_min=0.5, r_max=0.5)
    d, st = _density(pace, imgs, params=p)
    _check_density(d, st, imgs, r_min=0.5, r_max=0.5)
    for s, img in zip(st, imgs):
        assert s["r"] == 0.5 and (s["h_out"], s["w_out"]) == O.target_size(img.shape[0], img.shape[1], 0.5)
    _no_device_error(pace)


def _tokens_case(pace, lens, D, seed, zero_rows=(), params=None, sizes=None):
    rng = np.random.default_rng(seed)
    cu = np.concatenate([[0], np.cumsum(lens)]).astype(np.int32)
    # preview-like tokens: a shared direction plus per-token detail of varying strength
    base = rng.normal(size=D)
    T = base[None, :] * rng.uniform(0.5, 2.0, (cu[-1], 1)) + rng.normal(size=(cu[-1], D)) * rng.uniform(
        0.05, 1.5, (cu[-1], 1))
    T[list(zero_rows)] = 0.0
    Tb = synth.f32_to_bf16_bits(T.astype(np.float32))
    sizes = sizes or [(28 * (8 + 3 * b), 28 * (10 + 2 * b)) for b in range(len(lens))]
    H = [h for h, _ in sizes]
    W = [w for _, w in sizes]
    d, st = pace.pace_apc_density_tokens(bf16_tensor(Tb).view(-1, D), cu, H, W, params=params)
    return f64(Tb).reshape(-1, D), cu, H, W, d.cpu().numpy(), pace.stats_dict(st)


@pytest.mark.parametrize("lens,D", [([1024], 1280), ([37], 64), ([5000, 3, 200], 1152), ([700], 4096)])
def test_density_tokens(pace, lens, D):
    """Eq. 1-6 on preview tokens (the paper's own input) against the oracle."""
    T, cu, H, W, d, st = _tokens_case(pace, lens, D, seed=D + len(lens), zero_rows=[1] if lens[0] > 1 else [])
    for b in range(len(lens)):
        ref = O.apc_density_preview(T[cu[b]:cu[b + 1]], H[b], W[b])
        s = st[b]
        assert s["n_patches"] == lens[b] and s["k_tail"] == ref["k_tail"]
        assert_distances_close(d[cu[b]:cu[b + 1]], ref["d"], what="token d_i")
        for k in ("phi", "d_top", "rho_d", "r"):
            assert abs(s[k] - ref[k]) <= 2e-3 * max(abs(ref[k]), 1e-3), (k, s[k], ref[k])
        assert abs(s["rho"] - ref["rho"]) <= 2e-3 * max(abs(ref["rho"]), 1e-3) + 2e-6
        for side, key, exp in ((H[b], "h_out", ref["H_out"]), (W[b], "w_out", ref["W_out"])):
            x = side * math.sqrt(max(ref["r"], 0.0)) / 28 + 0.5
            assert s[key] == exp or (abs(x - round(x)) < 2e-3 * x and abs(s[key] - exp) == 28), (key, s[key], exp)
    _no_device_error(pace)


def test_density_tokens_params_and_rejects(pace):
    p = pace.apc_params(alpha=0.2, gamma=0.9, tail_frac=0.2, r_min=0.3, r_max=0.6)
    T, cu, H, W, d, st = _tokens_case(pace, [300, 41], 256, seed=5, params=p)
    for b in range(2):
        ref = O.apc_density_preview(T[cu[b]:cu[b + 1]], H[b], W[b], 0.2, 0.9, 0.2, 0.3, 0.6)
        assert abs(st[b]["r"] - ref["r"]) <= 2e-3 * ref["r"] and st[b]["k_tail"] == ref["k_tail"]
    Tt = torch.zeros((10, 63), dtype=torch.bfloat16, device="cuda")
    with pytest.raises(pace.PaceError):
        pace.pace_apc_density_tokens(Tt, [0, 10], [28], [28])           # odd D
    Tt = torch.zeros((10, 64), dtype=torch.bfloat16, device="cuda")
    with pytest.raises(pace.PaceError):
        pace.pace_apc_density_tokens(Tt, [0, 10, 10], [28, 28], [28, 28])   # an image without tokens


@pytest.mark.parametrize("feature", ["rgb_stats", "color_entropy", "edge_density", "laplacian"])
def test_pixel_features_and_density(pace, feature):
    """Pixel-statistic previews: the feature tokens, then Eq. 1-6 on them, against the oracle."""
    rng = np.random.default_rng(17)
    imgs = [synth.make_image(rng, h, w, 3, 2, f) for h, w, f in [(448, 448, 0.3), (70, 462, 0.6), (1008, 28, 0.1)]]
    imgs.append(np.full((56, 84, 3), 200, np.uint8))                         # a constant image
    buf, off = synth.pack_images(imgs)
    H = [im.shape[0] for im in imgs]
    W = [im.shape[1] for im in imgs]
    img_t = torch.from_numpy(buf).cuda()
    tok = pace.pace_apc_pixel_features(img_t, off, H, W, feature).cpu().numpy()
    d, st = pace.pace_apc_density_pixel(img_t, off, H, W, feature)
    d, st = d.cpu().numpy(), pace.stats_dict(st)
    p0 = 0
    dim = O.FEATURE_DIMS[feature]
    for im, s in zip(imgs, st):
        ref_tok = O.pixel_statistic_tokens(im, feature)
        n = ref_tok.shape[0]
        # integer-derived statistics: fp32 rounding only; the padding stays zero
        np.testing.assert_allclose(tok[p0:p0 + n, :dim], ref_tok, rtol=2e-6, atol=2e-6, err_msg=feature)
        assert not tok[p0:p0 + n, dim:].any()
        ref = O.apc_density_pixel(im, feature)
        assert s["n_patches"] == n and s["k_tail"] == ref["k_tail"]
        assert_distances_close(d[p0:p0 + n], ref["d"], what=f"d_i ({feature})")
        for k in ("phi", "d_top", "rho_d", "r"):
            assert abs(s[k] - ref[k]) <= 2e-3 * max(abs(ref[k]), 1e-3), (feature, k, s[k], ref[k])
        p0 += n
    _no_device_error(pace)


def test_pixel_features_rejects(pace):
    img = torch.zeros(28 * 28 * 3, dtype=torch.uint8, device="cuda")
    with pytest.raises(pace.PaceError):
        pace.pace_apc_pixel_features(img, [0], [28], [28], 4)          # unknown feature
    with pytest.raises(pace.PaceError):
        pace.pace_apc_density_pixel(img, [0], [28], [30], "laplacian")   # not a multiple of 14


def test_density_constant_images(pace):
    imgs = [np.full((112, 168, 3), v, dtype=np.uint8) for v in (0, 77, 255)]
    d, st = _density(pace, imgs)
    assert np.abs(d).max() < 2e-3
    for s in st:
        assert abs(s["phi"] - 1.0) < 1e-5 and abs(s["rho"]) < 2e-3
        assert (s["h_out"], s["w_out"]) == (28, 28)


def _background_with_noise(rng, side, noisy):
    img = np.full((side, side, 3), 120, dtype=np.uint8)
    g = side // 14
    for q in rng.choice(g * g, size=int(noisy * g * g), replace=False):
        y, x = divmod(int(q), g)
        img[14 * y:14 * y + 14, 14 * x:14 * x + 14] = rng.integers(0, 256, (14, 14, 3), dtype=np.uint8)
    return img


@pytest.mark.parametrize("side,noisy", [(1008, 0.05), (896, 0.03), (896, 0.5)])
def test_density_crowded_tail(pace, side, noisy):
    """Images whose tail bucket is crowded with identical distances: a constant background with
    a fraction of noise patches.  1008^2 at 5 % puts ~4900 equal distances in the k-th largest's
    bucket (more than the 4096-entry list: whole-array selection rounds); 896^2 at 3 % puts ~3970
    there (the compacted list, full of equal keys); 896^2 at 50 % has the k-th largest among the
    noise patches."""
    rng = np.random.default_rng(side + int(noisy * 100))
    img = _background_with_noise(rng, side, noisy)
    d, st = _density(pace, [img])
    _check_density(d, st, [img])
    _no_device_error(pace)


def test_density_tail_paths_mixed_in_one_call(pace):
    """The three ways the tail narrows the k-th largest distance, in one call: a crowded bucket
    (1008^2 at 5 % noise: more equal distances than the member list holds, narrowed over the
    whole array), a list full of equal keys (896^2 at 3 %: offset rounds over the list) and a
    short list (a natural image: direct ranking).  The images have 5184, 1056 and 4096 patches,
    i.e. 2, 1 and 1 CTAs of the tail, so each image's last CTA works beside the others.  Every
    image must be bit-equal to a call with that image alone, and equal to the oracle."""
    rng = np.random.default_rng(77)
    imgs = [_background_with_noise(rng, 1008, 0.05), synth.make_image(rng, 448, 462, 4, 4, 0.5),
            _background_with_noise(rng, 896, 0.03)]
    d, st = _density(pace, imgs)
    p0 = 0
    for b, im in enumerate(imgs):
        d1, st1 = _density(pace, [im])
        n = d1.size
        np.testing.assert_array_equal(d[p0:p0 + n], d1)
        assert st[b] == st1[0], b
        p0 += n
    _check_density(d, st, imgs)
    _no_device_error(pace)


def test_density_large_and_small_images_in_one_call(pace):
    """One image of 224 x 224 patches (50176: more distances than the tail stages in shared
    memory) next to a small one in the same call: every image must come out bit-equal to a call
    with that image alone, and the small one equal to the oracle."""
    rng = np.random.default_rng(31)
    big = synth.make_image(rng, 3136, 3136, 8, 8, 0.3)
    small = synth.make_image(rng, 448, 616, 4, 4, 0.5)
    d, st = _density(pace, [small, big])
    d_small, st_small = _density(pace, [small])
    d_big, st_big = _density(pace, [big])
    n_small = (448 // 14) * (616 // 14)
    np.testing.assert_array_equal(d[:n_small], d_small)
    np.testing.assert_array_equal(d[n_small:], d_big)
    assert st[0] == st_small[0] and st[1] == st_big[0]
    _check_density(d[:n_small], st[:1], [small])
    _no_device_error(pace)


def test_density_rejects_bad_sizes(pace):
    img = np.zeros((30, 28, 3), dtype=np.uint8)
    with pytest.raises(pace.PaceError) as e:
        _density(pace, [img])
    assert e.value.status == pace.PACE_ERR_INVALID_ARG


def _resample_gpu(pace, images, sizes):
    buf, off = synth.pack_images(images)
    H = [im.shape[0] for im in images]
    W = [im.shape[1] for im in images]
    dst_off = np.concatenate([[0], np.cumsum([h * w * 3 for h, w in zip(H, W)])])[:-1]
    dst = torch.zeros(int(sum(h * w * 3 for h, w in zip(H, W))), dtype=torch.uint8, device="cuda")
    pace.pace_apc_resample_to(torch.from_numpy(buf).cuda(), off, H, W, [s[0] for s in sizes],
                              [s[1] for s in sizes], dst, dst_off)
    out = dst.cpu().numpy()
    return [out[o:o + ho * wo * 3].reshape(ho, wo, 3) for o, (ho, wo) in zip(dst_off, sizes)]


@pytest.mark.parametrize("shape,size", [((56, 84), (28, 28)), ((98, 70), (42, 56)), ((140, 140), (28, 70)),
                                        ((84, 56), (37, 19)), ((448, 448), (308, 308)), ((56, 84), (56, 84)),
                                        ((616, 1232), (28, 28)), ((2156, 392), (1092, 196))])
def test_resample_within_one_lsb(pace, shape, size):
    rng = np.random.default_rng(shape[0] + size[1])
    img = synth.make_image(rng, shape[0], shape[1], 3, 3, 0.5)
    out = _resample_gpu(pace, [img], [size])[0]
    ref = O.apc_resample(img, *size)
    diff = np.abs(out.astype(np.int32) - ref.astype(np.int32))
    assert diff.max() <= 1, diff.max()
    if size == shape:
        np.testing.assert_array_equal(out, img)
    _no_device_error(pace)


def test_resample_constant_bit_exact_and_batch(pace):
    imgs = [np.full((112, 168, 3), v, dtype=np.uint8) for v in (0, 201, 255)]
    sizes = [(28, 28), (56, 84), (84, 112)]
    for o, v in zip(_resample_gpu(pace, imgs, sizes), (0, 201, 255)):
        assert np.all(o == v)
    rng = np.random.default_rng(5)
    imgs = [synth.make_image(rng, h, w, 2, 2, 0.5) for h, w in [(224, 448), (56, 56), (616, 532)]]
    sizes = [(112, 308), (28, 28), (420, 364)]
    for o, im, sz in zip(_resample_gpu(pace, imgs, sizes), imgs, sizes):
        assert np.abs(o.astype(int) - O.apc_resample(im, *sz).astype(int)).max() <= 1


def test_resample_from_device_stats(pace):
    """pace_apc_resample reads (h_out, w_out) on the device; same pixels as the explicit call."""
    rng = np.random.default_rng(6)
    imgs = [synth.make_image(rng, h, w, 4, 4, f) for h, w, f in [(448, 448, 0.5), (280, 560, 0.1)]]
    buf, off = synth.pack_images(imgs)
    H, W = [448, 280], [448, 560]
    src = torch.from_numpy(buf).cuda()
    _, st = pace.pace_apc_density(src, off, H, W)
    sd = pace.stats_dict(st)
    dst_off = [0, 448 * 448 * 3]
    dst = torch.zeros(448 * 448 * 3 + 280 * 560 * 3, dtype=torch.uint8, device="cuda")
    pace.pace_apc_resample(src, off, H, W, st, dst, dst_off)
    dst2 = torch.zeros_like(dst)
    pace.pace_apc_resample_to(src, off, H, W, [s["h_out"] for s in sd], [s["w_out"] for s in sd], dst2, dst_off)
    for b, s in enumerate(sd):
        n = s["h_out"] * s["w_out"] * 3
        assert torch.equal(dst[dst_off[b]:dst_off[b] + n], dst2[dst_off[b]:dst_off[b] + n])
        ref = O.apc_density(imgs[b])
        assert (s["h_out"], s["w_out"]) == (ref["H_out"], ref["W_out"])


# ----------------------------------------------------------------------------------------------
# attention importance
# ----------------------------------------------------------------------------------------------
def _vit_case(pace, lens, H=16, D=80, merge=4, seed=0, boost=None):
    cu = np.concatenate([[0], np.cumsum(lens)]).astype(np.int32)
    Qb = synth.random_small_qk(seed, int(cu[-1]), H, D)
    Kb = synth.random_small_qk(seed + 1000, int(cu[-1]), H, D)
    if boost is not None:        # a few rows with 4x norm (attention sinks)
        Kb = synth.f32_to_bf16_bits(f64(Kb).astype(np.float32) * boost[:, None, None].astype(np.float32))
    scale = 1.0 / math.sqrt(D)
    out = pace.pace_vit_attn_importance(bf16_tensor(Qb), bf16_tensor(Kb), cu, scale, merge).cpu().numpy()
    ref = O.vit_attn_importance(f64(Qb), f64(Kb), cu, scale, merge)
    return out, ref, cu


@pytest.mark.parametrize("lens", [[4], [64], [100], [128], [256], [300], [1024], [516, 4, 128, 388]])
def test_vit_importance(pace, lens):
    out, ref, cu = _vit_case(pace, lens)
    assert_scores_close(out, ref, what="S_vis_raw")
    for b in range(len(lens)):     # each image's map sums to N * heads
        assert out[cu[b] // 4:cu[b + 1] // 4].sum() == pytest.approx(lens[b] * 16, rel=1e-4)
    _no_device_error(pace)


@pytest.mark.parametrize("D,H,merge", [(64, 4, 1), (128, 2, 2), (80, 3, 1)])
def test_vit_importance_head_dims(pace, D, H, merge):
    out, ref, _ = _vit_case(pace, [200, 36], H=H, D=D, merge=merge, seed=D)
    assert_scores_close(out, ref, what=f"S_vis_raw D={D}")


def test_vit_importance_sinks(pace):
    n = 384
    boost = np.ones(n)
    boost[[5, 77, 300]] = 4.0
    out, ref, _ = _vit_case(pace, [n], boost=boost, seed=11)
    assert_scores_close(out, ref, what="S_vis_raw with sinks")


def _spiked_qk(n, H, D, seed, spikes):
    """Random Q/K with planted score spikes: for (key, rows, norm) the key and the query rows
    get the same direction u with length `norm`, so those rows score norm^2 against that key,
    far above everything before it in the row."""
    rng = np.random.default_rng(seed)
    Q = f64(synth.random_small_qk(seed, n, H, D))
    K = f64(synth.random_small_qk(seed + 1000, n, H, D))
    for key, rows, norm in spikes:
        u = rng.standard_normal((H, D))
        u /= np.linalg.norm(u, axis=1, keepdims=True)
        K[key] = norm * u
        Q[rows] = norm * u + 0.05 * rng.standard_normal((len(rows), H, D))
    return (synth.f32_to_bf16_bits(Q.astype(np.float32)), synth.f32_to_bf16_bits(K.astype(np.float32)))


def test_vit_importance_wide_score_range(pace):
    """Rows whose maximum lies 88 and 244 (base 2) above the scores of their first keys: the
    first stays finite in the fixed-shift sum (shift = first maximum + 90), the second overflows
    it and the CTA streams its keys again with an exact running maximum."""
    n, H, D = 1024, 2, 80
    Qb, Kb = _spiked_qk(n, H, D, seed=5, spikes=[(700, np.arange(0, 200), 25.0),
                                                 (900, np.arange(300, 340), 40.0)])
    cu = np.array([0, n], np.int32)
    scale = 1.0 / math.sqrt(D)
    out = pace.pace_vit_attn_importance(bf16_tensor(Qb), bf16_tensor(Kb), cu, scale, 1).cpu().numpy()
    ref = O.vit_attn_importance(f64(Qb), f64(Kb), cu, scale, 1)
    assert ref[700] > 150 and ref[900] > 30       # the spikes dominate their rows
    assert_scores_close(out, ref, what="S_vis_raw with score spikes")
    _no_device_error(pace)


def test_vit_importance_high_run_below_margin(pace):
    """Rows whose 7936 last keys all score about 91 (base 2) above their first keys: the warps
    that start on the low keys hold the high terms just below the fixed shift's margin (no
    overflow, no redo) while the first keys' terms sit near 2^-90."""
    n, H, D, a = 8192, 1, 80, 24.6
    rng = np.random.default_rng(11)
    Q = f64(synth.random_small_qk(11, n, H, D))
    K = f64(synth.random_small_qk(1011, n, H, D))
    u = rng.standard_normal((H, D))
    u /= np.linalg.norm(u, axis=1, keepdims=True)
    K[256:] = a * u
    Q[:64] = a * u + 0.05 * rng.standard_normal((64, H, D))
    Qb, Kb = synth.f32_to_bf16_bits(Q.astype(np.float32)), synth.f32_to_bf16_bits(K.astype(np.float32))
    cu = np.array([0, n], np.int32)
    scale = 1.0 / math.sqrt(D)
    out = pace.pace_vit_attn_importance(bf16_tensor(Qb), bf16_tensor(Kb), cu, scale, 1).cpu().numpy()
    ref = O.vit_attn_importance(f64(Qb), f64(Kb), cu, scale, 1)
    assert_scores_close(out, ref, what="S_vis_raw with a long run of high scores")
    _no_device_error(pace)


@pytest.mark.parametrize("ends", ["auto1", "auto3", "auto7", "ragged"])
def test_vit_importance_chunked_matches_unchunked(pace, ends):
    """The row pass split by query rows, each piece after an event that marks its Q rows copied
    in on a side stream, gives the same bits as the one-launch call.  Q starts as NaN, so a piece
    that read rows not yet copied would show up unless those rows are only past its images."""
    lens = [516, 4, 128, 1300, 388, 2052]
    H, D, merge = 16, 80, 4
    cu = np.concatenate([[0], np.cumsum(lens)]).astype(np.int32)
    total = int(cu[-1])
    Qb = synth.random_small_qk(21, total, H, D)
    Kb = synth.random_small_qk(1021, total, H, D)
    spike = np.zeros((total,), np.float32)
    spike[[40, 700, 2000]] = 9.0              # three query rows with 10x norm
    Qb = synth.f32_to_bf16_bits(f64(Qb).astype(np.float32) * (1 + spike[:, None, None]))
    Q, K = bf16_tensor(Qb), bf16_tensor(Kb)
    scale = 1.0 / math.sqrt(D)
    want = pace.pace_vit_attn_importance(Q, K, cu, scale, merge)
    if ends == "ragged":
        e = np.array([37, 37, 900, 2500, total], np.int64)    # unaligned, with an empty piece
    else:
        e = pace.vit_chunk_rows(cu, int(ends[4:]))
    assert e[-1] == total and np.all(np.diff(e) >= 0)
    host = Q.cpu().pin_memory()
    dq = torch.full_like(Q, float("nan"))
    side = torch.cuda.Stream()
    side.wait_stream(torch.cuda.current_stream())
    evs, r0 = [], 0
    with torch.cuda.stream(side):
        for r1 in e:
            dq[r0:r1].copy_(host[r0:r1], non_blocking=True)
            ev = torch.cuda.Event()
            ev.record(side)
            evs.append(ev)
            r0 = int(r1)
    got = pace.pace_vit_attn_importance_chunked(dq, K, cu, e, evs, scale, merge)
    torch.cuda.synchronize()
    assert torch.equal(got, want)
    ref = O.vit_attn_importance(f64(Qb), f64(Kb), cu, scale, merge)
    assert_scores_close(got.cpu().numpy(), ref, what="chunked S_vis_raw")
    _no_device_error(pace)


def test_vit_importance_nan_rows_stay_in_their_image(pace):
    """NaN and inf in the query rows of some images of a ragged batch: every other image's
    S_vis_raw still equals the oracle's on its own (clean) rows.  An image's last query tile
    in pass 2 also covers the next image's first rows; those columns are masked explicitly."""
    lens = [300, 516, 4, 1300, 388, 260]
    H, D, merge = 4, 80, 4
    cu = np.concatenate([[0], np.cumsum(lens)]).astype(np.int32)
    total = int(cu[-1])
    Qb = synth.random_small_qk(31, total, H, D)
    Kb = synth.random_small_qk(1031, total, H, D)
    scale = 1.0 / math.sqrt(D)
    ref = O.vit_attn_importance(f64(Qb), f64(Kb), cu, scale, merge)
    Q = bf16_tensor(Qb)
    Q[cu[1]:cu[1] + 7] = float("nan")            # image 1: its first rows (inside image 0's last tile)
    Q[cu[3]] = float("inf")                       # image 3: first row +inf, another row -inf
    Q[cu[3] + 1, :, 5] = float("-inf")
    Q[cu[5]:cu[6]] = float("nan")                 # image 5: every row, past the end of image 4
    out = pace.pace_vit_attn_importance(Q, bf16_tensor(Kb), cu, scale, merge).cpu().numpy()
    for b in (0, 2, 4):
        m0, m1 = cu[b] // merge, cu[b + 1] // merge
        assert np.isfinite(out[m0:m1]).all(), b
        assert_scores_close(out[m0:m1], ref[m0:m1], what=f"S_vis_raw of clean image {b}")
    _no_device_error(pace)


def test_llm_importance_nan_queries_stay_in_their_image(pace):
    """The same isolation on the LLM text->visual path (GQA): NaN text queries of image 1 leave
    images 0 and 2 equal to the oracle."""
    tq, nv = [70, 33, 140], [300, 129, 260]
    Hq, Hkv, D = 8, 2, 128
    cu_q = np.concatenate([[0], np.cumsum(tq)]).astype(np.int32)
    cu_k = np.concatenate([[0], np.cumsum(nv)]).astype(np.int32)
    Qb = synth.random_small_qk(41, int(cu_q[-1]), Hq, D)
    Kb = synth.random_small_qk(1041, int(cu_k[-1]), Hkv, D)
    scale = 1.0 / math.sqrt(D)
    ref = O.llm_text_visual_importance(f64(Qb), f64(Kb), cu_q, cu_k, scale)
    Q = bf16_tensor(Qb)
    Q[cu_q[1]:cu_q[2]] = float("nan")
    out = pace.pace_llm_text_visual_importance(Q, bf16_tensor(Kb), cu_q, cu_k, scale).cpu().numpy()
    for b in (0, 2):
        v0, v1 = cu_k[b], cu_k[b + 1]
        assert np.isfinite(out[v0:v1]).all(), b
        assert_scores_close(out[v0:v1], ref[v0:v1], what=f"S_llm_raw of clean image {b}")
    _no_device_error(pace)


def test_vit_importance_chunked_rejects_bad_chunks(pace):
    Q = torch.zeros((8, 1, 64), dtype=torch.bfloat16, device="cuda")
    ev = torch.cuda.Event()
    ev.record()
    with pytest.raises(pace.PaceError):
        pace.pace_vit_attn_importance_chunked(Q, Q, [0, 8], [4], [ev], merge=4)       # last end != total
    with pytest.raises(pace.PaceError):
        pace.pace_vit_attn_importance_chunked(Q, Q, [0, 8], [6, 4, 8], [ev, ev, ev], merge=4)   # decreasing
    with pytest.raises(ValueError):
        pace.pace_vit_attn_importance_chunked(Q, Q, [0, 8], [4, 8], [ev], merge=4)    # one event per chunk


def test_llm_importance_wide_score_range(pace):
    """A spike about 245 (base 2) above the other scores through the GQA path with key splits
    (few query tiles, many key tiles): the fixed-shift sum overflows in every split that holds
    the spike key, which redoes its keys with an exact running maximum."""
    nq, nk, Hq, Hkv, D = 64, 2304, 4, 2, 128
    Qs, _ = _spiked_qk(nq, Hq, D, seed=6, spikes=[])
    rng = np.random.default_rng(6)
    Q = f64(Qs)
    K = f64(synth.random_small_qk(7, nk, Hkv, D))
    for g in range(Hkv):
        u = rng.standard_normal(D)
        u /= np.linalg.norm(u)
        K[2000, g] = 44.0 * u
        for h in range(g * (Hq // Hkv), (g + 1) * (Hq // Hkv)):
            Q[:32, h] = 44.0 * u
    Qb, Kb = synth.f32_to_bf16_bits(Q.astype(np.float32)), synth.f32_to_bf16_bits(K.astype(np.float32))
    cq, ck = np.array([0, nq], np.int32), np.array([0, nk], np.int32)
    scale = 1.0 / math.sqrt(D)
    out = pace.pace_llm_text_visual_importance(bf16_tensor(Qb), bf16_tensor(Kb), cq, ck, scale).cpu().numpy()
    ref = O.llm_text_visual_importance(f64(Qb), f64(Kb), cq, ck, scale)
    assert ref[2000] > 32 * Hq * 0.9
    assert_scores_close(out, ref, what="S_llm_raw with score spikes")
    _no_device_error(pace)


def _llm_case(pace, tq, nv, Hq=28, Hkv=4, D=128, seed=0):
    cq = np.concatenate([[0], np.cumsum(tq)]).astype(np.int32)
    ck = np.concatenate([[0], np.cumsum(nv)]).astype(np.int32)
    Qb = synth.random_small_qk(seed, int(cq[-1]), Hq, D)
    Kb = synth.random_small_qk(seed + 1, int(ck[-1]), Hkv, D)
    scale = 1.0 / math.sqrt(D)
    out = pace.pace_llm_text_visual_importance(bf16_tensor(Qb), bf16_tensor(Kb), cq, ck, scale).cpu().numpy()
    ref = O.llm_text_visual_importance(f64(Qb), f64(Kb), cq, ck, scale)
    return out, ref, cq, ck


@pytest.mark.parametrize("tq,nv", [([64], [256]), ([1], [1]), ([5], [300]), ([130], [129]), ([256], [2304]),
                                   ([32, 200, 77], [100, 640, 3])])
def test_llm_importance(pace, tq, nv):
    out, ref, cq, ck = _llm_case(pace, tq, nv)
    assert_scores_close(out, ref, what="S_llm_raw")
    for b in range(len(tq)):
        assert out[ck[b]:ck[b + 1]].sum() == pytest.approx(tq[b] * 28, rel=1e-4)
    _no_device_error(pace)


def test_llm_importance_gqa_shapes(pace):
    for Hq, Hkv, D in ((8, 8, 64), (12, 2, 80), (4, 1, 128)):
        out, ref, _, _ = _llm_case(pace, [40, 9], [70, 260], Hq=Hq, Hkv=Hkv, D=D, seed=Hq)
        assert_scores_close(out, ref, what=f"S_llm_raw Hq={Hq} Hkv={Hkv}")


def _seq_case(pace, S, vis, nvis, query_set, Hq=28, Hkv=4, D=128, seed=0):
    cu = np.concatenate([[0], np.cumsum(S)]).astype(np.int32)
    Qb = synth.random_small_qk(seed, int(cu[-1]), Hq, D)
    Kb = synth.random_small_qk(seed + 1, int(cu[-1]), Hkv, D)
    scale = 1.0 / math.sqrt(D)
    out = pace.pace_llm_sequence_importance(bf16_tensor(Qb), bf16_tensor(Kb), cu, vis, nvis, query_set,
                                            scale).cpu().numpy()
    ref = O.llm_sequence_importance(f64(Qb), f64(Kb), cu, vis, nvis, scale, query_set)
    return out, ref


@pytest.mark.parametrize("query_set", ["vision_text", "text", "last"])
@pytest.mark.parametrize("S,vis,nvis", [([700], [30], [400]), ([1300], [3], [1024]), ([9], [2], [4])])
def test_llm_sequence_importance(pace, S, vis, nvis, query_set):
    out, ref = _seq_case(pace, S, vis, nvis, query_set)
    assert_scores_close(out, ref, what=f"full-sequence S_llm_raw ({query_set})")
    _no_device_error(pace)


@pytest.mark.parametrize("query_set", ["vision_text", "text", "last"])
def test_llm_sequence_importance_ragged_gqa(pace, query_set):
    # the first sequence ends with its visual span, so its text query set is empty
    S, vis, nvis = [300, 1100, 77, 520], [0, 14, 5, 200], [300, 900, 60, 1]
    for Hq, Hkv, D in ((8, 2, 80), (12, 12, 64)):
        out, ref = _seq_case(pace, S, vis, nvis, query_set, Hq=Hq, Hkv=Hkv, D=D, seed=Hq)
        assert_scores_close(out, ref, what=f"full-sequence S_llm_raw ({query_set}, Hq={Hq}, Hkv={Hkv})")
        if query_set == "text":
            assert np.all(out[:300] == 0.0)
    _no_device_error(pace)


def test_llm_sequence_importance_all_visual_mass(pace):
    # an all-visual sequence: every query row's causal softmax lies on visual keys
    out, _ = _seq_case(pace, [640, 257], [0, 0], [640, 257], "vision_text", Hq=4, Hkv=1, D=64, seed=5)
    assert out[:640].sum() == pytest.approx(640 * 4, rel=1e-4)
    assert out[640:].sum() == pytest.approx(257 * 4, rel=1e-4)
    # key 0 is seen by every row; the last key only by the last row (weight of its own softmax)
    assert out[639] < out[0]


def test_llm_sequence_importance_rejects(pace):
    Q = torch.zeros((16, 2, 64), dtype=torch.bfloat16, device="cuda")
    for cu, vis, nvis, qs in (([0, 16], [10], [7], "vision_text"),     # visual span past the end
                              ([0, 16], [-1], [4], "text"),            # negative start
                              ([0, 16], [0], [0], "last"),             # no visual tokens
                              ([0, 16], [0], [4], 7)):                  # unknown query set
        with pytest.raises(pace.PaceError):
            pace.pace_llm_sequence_importance(Q, Q, cu, vis, nvis, qs)
    _no_device_error(pace)


def test_importance_rejects_bad_args(pace):
    Q = torch.zeros((8, 2, 80), dtype=torch.bfloat16, device="cuda")
    with pytest.raises(pace.PaceError):
        pace.pace_vit_attn_importance(Q, Q, [0, 6], merge=4)          # 6 % 4 != 0
    with pytest.raises(pace.PaceError):
        pace.pace_vit_attn_importance(Q, Q, [0, 0, 8], merge=4)       # empty image
    Q = torch.zeros((8, 2, 72), dtype=torch.bfloat16, device="cuda")
    with pytest.raises(pace.PaceError):
        pace.pace_vit_attn_importance(Q, Q, [0, 8], merge=4)          # head_dim 72


# ----------------------------------------------------------------------------------------------
# DDAE select
# ----------------------------------------------------------------------------------------------
def _select(pace, sl, sv, cu, keep, tau=0.5, fusion=0):
    r = pace.pace_ddae_select(torch.from_numpy(sl.astype(np.float32)).cuda(),
                              torch.from_numpy(sv.astype(np.float32)).cuda(), cu,
                              np.concatenate([[0], np.cumsum(keep)]).astype(np.int32),
                              pace.ddae_params(tau=tau, fusion=fusion))
    return [x.cpu().numpy() for x in r]


@pytest.mark.parametrize("mode,name", [(1, "only_llm"), (2, "only_vit"), (3, "fixed")])
def test_ddae_fusion_ablations(pace, mode, name):
    """The fusion ablations (Only LLM-Attn, Only ViT-Attn, Fixed Fusion) against the oracle."""
    rng = np.random.default_rng(40 + mode)
    lens = [300, 2584, 17]
    cu = np.concatenate([[0], np.cumsum(lens)]).astype(np.int32)
    sl = rng.gamma(0.5, 2.0, size=cu[-1]).astype(np.float32)
    sv = rng.lognormal(0, 1, size=cu[-1]).astype(np.float32)
    keep = [O.budget(n, 0.1) for n in lens]
    s_final, w, kept = _select(pace, sl, sv, cu, keep, fusion=mode)
    k0 = 0
    for b, n in enumerate(lens):
        v0, v1 = cu[b], cu[b + 1]
        f = O.ddae_fuse(sl[v0:v1].astype(np.float64), sv[v0:v1].astype(np.float64), fusion=name)
        assert (w[b, 0], w[b, 1]) == O.FUSION_WEIGHTS[name]
        assert_scores_close(s_final[v0:v1], f["S_final"], atol_frac=2e-3, what=f"S_final {name}")
        assert_kept_matches(kept[k0:k0 + keep[b]], f["S_final"], keep[b], offset=v0)
        k0 += keep[b]
    with pytest.raises(pace.PaceError):
        _select(pace, sl, sv, cu, keep, fusion=4)
    _no_device_error(pace)


@pytest.mark.parametrize("lens,fracs", [([256], [0.1]), ([2584], [0.1]), ([10549], [0.05]), ([1], [1.0]),
                                        ([7, 300, 1000, 24576], [0.25, 0.0, 1.0, 0.1]),
                                        ([4096, 4097, 12288, 12289], [0.1, 0.05, 0.25, 0.1]),
                                        ([42196], [0.1]), ([150000, 3], [0.02, 0.5])])
def test_ddae_select_random(pace, lens, fracs):
    rng = np.random.default_rng(len(lens) + lens[0])
    cu = np.concatenate([[0], np.cumsum(lens)]).astype(np.int32)
    sl = rng.gamma(0.5, 2.0, size=cu[-1]).astype(np.float32)
    sv = rng.lognormal(0, 1, size=cu[-1]).astype(np.float32)
    keep = [O.budget(n, f) for n, f in zip(lens, fracs)]
    s_final, w, kept = _select(pace, sl, sv, cu, keep)
    k0 = 0
    for b, n in enumerate(lens):
        v0, v1 = cu[b], cu[b + 1]
        f = O.ddae_fuse(sl[v0:v1].astype(np.float64), sv[v0:v1].astype(np.float64))
        assert_scores_close(s_final[v0:v1], f["S_final"], atol_frac=2e-3, what="S_final")
        assert abs(w[b, 0] - f["alpha_w"]) < 2e-3 * f["alpha_w"] and abs(w[b, 1] - f["beta_w"]) < 2e-3 * f["beta_w"]
        assert_kept_matches(kept[k0:k0 + keep[b]], f["S_final"], keep[b], offset=v0)
        k0 += keep[b]


def test_ddae_select_exact_decisions_with_ties(pace):
    """S_llm == S_vis with min 0 and max 1: S_final = x exactly in fp32 and fp64, so the kept
    set (ties broken by the lower index) must equal the oracle's bit for bit."""
    rng = np.random.default_rng(9)
    for n, K in ((1000, 100), (4096, 1), (333, 332), (50, 25), (20000, 2000), (12289, 7)):
        x = np.round(rng.uniform(size=n) * 16) / 16      # many exact ties
        x[0], x[-1] = 0.0, 1.0
        cu = np.array([0, n], dtype=np.int32)
        s_final, w, kept = _select(pace, x, x, cu, [K])
        np.testing.assert_array_equal(s_final, x.astype(np.float32))
        assert w[0, 0] == 0.5 and w[0, 1] == 0.5
        np.testing.assert_array_equal(kept, O.top_k_ascending(x, K))


def test_ddae_select_golden_and_constant(pace, golden):
    g = golden("ddae_four_tokens.txt")
    sl, sv = np.array(g["s_llm_raw"]), np.array(g["s_vis_raw"])
    s_final, w, kept = _select(pace, sl, sv, np.array([0, 4], np.int32), [2])
    np.testing.assert_allclose(s_final, g["s_final"], atol=1e-6)
    np.testing.assert_allclose(w[0], [g["alpha_w"], g["beta_w"]], atol=1e-6)
    assert kept.tolist() == [int(v) for v in g["kept_top2"]]
    s_final, w, kept = _select(pace, np.full(10, 3.0), np.arange(10.0), np.array([0, 10], np.int32), [3])
    assert kept.tolist() == [7, 8, 9]
    # both maps constant: S_final = 0 everywhere, every score ties, the lowest indices are kept
    for n in (10, 5000, 13000):
        s_final, w, kept = _select(pace, np.full(n, 2.0), np.full(n, 7.0), np.array([0, n], np.int32), [3])
        assert not s_final.any() and kept.tolist() == [0, 1, 2]


def test_ddae_select_non_finite_scores_are_reported(pace):
    """A NaN or inf raw score records PACE_ERR_INVALID_ARG (kernel id 9) in the device status
    word.  The map's scores are then not meaningful (NaN reaches the Eq. 7 weights), but the call
    still writes K distinct in-range indices in ascending order, the same on every run."""
    n = 600
    rng = np.random.default_rng(3)
    sl = rng.uniform(size=n).astype(np.float32)
    sv = rng.uniform(size=n).astype(np.float32)
    sl[[10, 500]] = np.nan
    for bad_v in (None, np.inf):
        if bad_v is not None:
            sl[[10, 500]] = 0.5
            sv[7] = bad_v
        outs = []
        for _ in range(2):
            _, _, kept = _select(pace, sl, sv, np.array([0, n], np.int32), [n // 3])
            code, where = pace.pace_device_status(clear=True)
            assert code == pace.PACE_ERR_INVALID_ARG and where == 9
            assert kept.size == n // 3 and np.all(np.diff(kept) > 0) and kept.min() >= 0 and kept.max() < n
            outs.append(kept)
        np.testing.assert_array_equal(outs[0], outs[1])


def test_ddae_select_rejects(pace):
    with pytest.raises(pace.PaceError):
        _select(pace, np.zeros(5), np.zeros(5), np.array([0, 5], np.int32), [6])
    with pytest.raises(pace.PaceError):
        _select(pace, np.zeros(5), np.zeros(5), np.array([0, 0, 5], np.int32), [0, 1])   # an empty map


# ----------------------------------------------------------------------------------------------
# prune step: row list and multi-tensor gather
# ----------------------------------------------------------------------------------------------
def test_prune_index_and_gather_multi(pace):
    """Pruned LLM context of a batch: row list from the kept tokens, then hidden states,
    KV-cache rows of two layers and M-RoPE position ids gathered in one launch (byte-exact)."""
    rng = np.random.default_rng(77)
    n_vis, pre, post = [300, 17, 1024], [40, 5, 0], [12, 0, 33]
    cu_vis = np.concatenate([[0], np.cumsum(n_vis)]).astype(np.int32)
    K = [O.budget(n, 0.1) for n in n_vis]
    cu_keep = np.concatenate([[0], np.cumsum(K)]).astype(np.int32)
    sl = rng.gamma(0.5, 2.0, cu_vis[-1]).astype(np.float32)
    sv = rng.lognormal(0, 1, cu_vis[-1]).astype(np.float32)
    _, _, kept = pace.pace_ddae_select(torch.from_numpy(sl).cuda(), torch.from_numpy(sv).cuda(), cu_vis, cu_keep)
    n_pre = [a + b + c for a, b, c in zip(pre, n_vis, post)]
    cu_seq = np.concatenate([[0], np.cumsum(n_pre)]).astype(np.int32)
    idx = pace.pace_prune_index(cu_seq, pre, cu_vis, cu_keep, kept)
    kept_h = kept.cpu().numpy()
    ref = np.concatenate([O.prune_rows(n_pre[b], pre[b], n_vis[b], kept_h[cu_keep[b]:cu_keep[b + 1]] - cu_vis[b])
                          + cu_seq[b] for b in range(3)])
    np.testing.assert_array_equal(idx.cpu().numpy(), ref)
    S, n = int(cu_seq[-1]), len(ref)
    hid = torch.randn(S, 896, device="cuda").to(torch.bfloat16)               # hidden states [S, D]
    kv = torch.randn(2, 2, 4, S, 128, device="cuda").to(torch.bfloat16)       # [layer, K/V, head, S, d]
    pos = torch.randint(0, 1 << 20, (3, S), device="cuda", dtype=torch.int64)  # M-RoPE ids [3, S]
    odd = torch.randint(0, 255, (S, 7), device="cuda", dtype=torch.uint8)     # 7-byte rows: byte path
    outs = [torch.empty(n, 896, dtype=torch.bfloat16, device="cuda"),
            torch.empty(2, 2, 4, n, 128, dtype=torch.bfloat16, device="cuda"),
            torch.empty(3, n, dtype=torch.int64, device="cuda"), torch.empty(n, 7, dtype=torch.uint8, device="cuda")]
    specs = [pace.gather_spec(hid, outs[0], 0), pace.gather_spec(kv, outs[1], 3), pace.gather_spec(pos, outs[2], 1),
             pace.gather_spec(odd, outs[3], 0)]
    pace.pace_gather_multi(specs, idx)
    r = torch.from_numpy(ref).cuda().long()
    assert torch.equal(outs[0], hid[r]) and torch.equal(outs[1], kv[:, :, :, r]) and torch.equal(outs[2], pos[:, r])
    assert torch.equal(outs[3], odd[r])
    _no_device_error(pace)
    bad = torch.tensor([0, S + 5], dtype=torch.int32, device="cuda")           # out of range: zero row + status
    o2 = torch.full((2, 896), 7, dtype=torch.bfloat16, device="cuda")
    pace.pace_gather_multi([pace.gather_spec(hid, o2, 0)], bad)
    torch.cuda.synchronize()
    code, where = pace.pace_device_status(clear=True)
    assert code == 1 and where == 13
    assert torch.equal(o2[0], hid[0]) and bool((o2[1] == 0).all())


# ----------------------------------------------------------------------------------------------
# batches larger than one kernel-parameter table (the host loops over groups of images)
# ----------------------------------------------------------------------------------------------
def test_many_images_attention(pace):
    """70 images: the attention calls take 64 images per launch table, so this runs two groups
    (ViT one-launch and in query-row pieces, LLM text -> visual)."""
    rng = np.random.default_rng(70)
    lens = [4 * int(x) for x in rng.integers(1, 40, 70)]
    out, ref, cu = _vit_case(pace, lens, H=4, merge=4, seed=70)
    assert_scores_close(out, ref, what="S_vis_raw, 70 images")
    Qb = synth.random_small_qk(70, int(cu[-1]), 4, 80)
    Kb = synth.random_small_qk(1070, int(cu[-1]), 4, 80)
    Q, K = bf16_tensor(Qb), bf16_tensor(Kb)
    scale = 1.0 / math.sqrt(80)
    want = pace.pace_vit_attn_importance(Q, K, cu, scale, 4)
    e = pace.vit_chunk_rows(cu, 5)
    evs = []
    for _ in e:
        ev = torch.cuda.Event()
        ev.record()
        evs.append(ev)
    got = pace.pace_vit_attn_importance_chunked(Q, K, cu, e, evs, scale, 4)
    torch.cuda.synchronize()
    assert torch.equal(got, want)
    tq = [int(x) for x in rng.integers(1, 20, 70)]
    nv = [int(x) for x in rng.integers(1, 90, 70)]
    out, ref, _, _ = _llm_case(pace, tq, nv, Hq=8, Hkv=2, seed=71)
    assert_scores_close(out, ref, what="S_llm_raw, 70 images")
    _no_device_error(pace)


def test_many_images_density_and_select(pace):
    """70 images through the density (64 per table), resample from the device statistics, and
    70 maps through fusion + top-K."""
    rng = np.random.default_rng(71)
    imgs = [synth.make_image(rng, 28 * int(h), 28 * int(w), 2, 2, float(f))
            for h, w, f in zip(rng.integers(1, 6, 70), rng.integers(1, 6, 70), rng.uniform(0.1, 0.9, 70))]
    d, st = _density(pace, imgs)
    _check_density(d, st, imgs)
    lens = [int(x) for x in rng.integers(1, 400, 70)]
    fracs = [float(x) for x in rng.choice([0.05, 0.1, 0.25, 1.0], 70)]
    cu = np.concatenate([[0], np.cumsum(lens)]).astype(np.int32)
    sl = rng.gamma(0.5, 2.0, size=cu[-1]).astype(np.float32)
    sv = rng.lognormal(0, 1, size=cu[-1]).astype(np.float32)
    keep = [O.budget(n, f) for n, f in zip(lens, fracs)]
    s_final, w, kept = _select(pace, sl, sv, cu, keep)
    k0 = 0
    for b, n in enumerate(lens):
        v0, v1 = cu[b], cu[b + 1]
        f = O.ddae_fuse(sl[v0:v1].astype(np.float64), sv[v0:v1].astype(np.float64))
        assert_scores_close(s_final[v0:v1], f["S_final"], atol_frac=2e-3, what="S_final, 70 maps")
        assert_kept_matches(kept[k0:k0 + keep[b]], f["S_final"], keep[b], offset=v0)
        k0 += keep[b]
    _no_device_error(pace)


def test_many_images_resample_tokens_sequences(pace):
    """70 images through the resample (target sizes read on the device), the preview-token
    density and the full-sequence S_llm: each takes 64 images per parameter table."""
    rng = np.random.default_rng(72)
    imgs = [synth.make_image(rng, 28 * int(h), 28 * int(w), 2, 2, float(f))
            for h, w, f in zip(rng.integers(1, 5, 70), rng.integers(1, 5, 70), rng.uniform(0.1, 0.9, 70))]
    buf, off = synth.pack_images(imgs)
    H = [im.shape[0] for im in imgs]
    W = [im.shape[1] for im in imgs]
    src = torch.from_numpy(buf).cuda()
    _, st = pace.pace_apc_density(src, off, H, W)
    sd = pace.stats_dict(st)
    dst_off = np.concatenate([[0], np.cumsum([h * w * 3 for h, w in zip(H, W)])])[:-1].astype(np.int64)
    dst = torch.zeros(int(sum(h * w * 3 for h, w in zip(H, W))), dtype=torch.uint8, device="cuda")
    pace.pace_apc_resample(src, off, H, W, st, dst, dst_off)
    flat = dst.cpu().numpy()
    for b, (img, s) in enumerate(zip(imgs, sd)):
        ho, wo = s["h_out"], s["w_out"]
        mine = flat[dst_off[b]:dst_off[b] + ho * wo * 3].reshape(ho, wo, 3).astype(np.int32)
        assert np.abs(mine - O.apc_resample(img, ho, wo).astype(np.int32)).max() <= 1, b
    lens = [int(x) for x in rng.integers(1, 60, 70)]
    T, cu, Ht, Wt, d, stt = _tokens_case(pace, lens, 64, seed=72, sizes=[(28 * 4, 28 * 4)] * 70)
    for b in range(70):
        ref = O.apc_density_preview(T[cu[b]:cu[b + 1]], Ht[b], Wt[b])
        assert_distances_close(d[cu[b]:cu[b + 1]], ref["d"], what="token d_i, 70 images")
    S = [int(x) for x in rng.integers(12, 80, 70)]
    vis = [int(rng.integers(0, s // 3)) for s in S]
    nvis = [int(rng.integers(1, s - v)) for s, v in zip(S, vis)]
    out, ref = _seq_case(pace, S, vis, nvis, "vision_text", Hq=8, Hkv=2, seed=72)
    assert_scores_close(out, ref, what="full-sequence S_llm_raw, 70 sequences")
    _no_device_error(pace)
