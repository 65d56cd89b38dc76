"""Full-size parity of the whole hot path on every benchmark workload.

Each workload (448x448, 1344x1344, 1904x1064 with sinks, 3836x2156, and the ragged
batch of 16 images) runs through HotPath, i.e. exactly the libpace calls and launch
configuration that bench.py times, and every output is compared with the fp64 oracle
computed at the same full size (the attention maps are fanned out over a spawn pool,
one (image, head) per job).
"""
import math

import numpy as np
import pytest
import torch

from oracle import pace_oracle as O
from paper_2608_27206_gb300 import synth
from tests.helpers import (assert_distances_close, assert_kept_matches, assert_scores_close, f64, oracle_vit,
                           spawn_pool)

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def pool():
    p = spawn_pool()
    yield p
    p.close()
    p.join()


@pytest.fixture(scope="module")
def pace():
    from paper_2608_27206_gb300 import build
    build.build()
    from paper_2608_27206_gb300 import pace as P
    P.pace_init(0)
    P.pace_device_status(clear=True)
    return P


def _near_half(x, rel=2e-3):
    return abs(x - math.floor(x) - 0.5) < rel * max(abs(x), 1.0)


@pytest.mark.parametrize("name", ["img448", "img1344", "frame1904", "img4k", "ragged16"])
def test_workload_full_size(pace, pool, name):
    from paper_2608_27206_gb300.hotpath import HotPath
    wl = synth.make_workload(name, seed=0)
    hp = HotPath(wl, "cuda")
    hp.step()
    torch.cuda.synchronize()
    code, where = pace.pace_device_status(clear=True)
    assert code == 0, (code, where)

    # --- condense: density statistics, distances, target sizes ---------------------------------
    d = hp.dist.cpu().numpy()
    stats = pace.stats_dict(hp.stats[: wl.B])
    p0 = 0
    oracle_sizes = []
    for b, (img, s) in enumerate(zip(wl.images, stats)):
        ref = O.apc_density(img)
        oracle_sizes.append((ref["H_out"], ref["W_out"]))
        n = ref["N"]
        assert s["n_patches"] == n and s["k_tail"] == ref["k_tail"]
        assert_distances_close(d[p0:p0 + n], ref["d"], what=f"{name}[{b}] d_i")
        for k in ("phi", "d_top", "rho_d", "rho", "r"):
            assert abs(s[k] - ref[k]) <= 2e-3 * max(abs(ref[k]), 1e-3) + 2e-6, (name, b, k, s[k], ref[k])
        for side, key, exp in ((img.shape[0], "h_out", ref["H_out"]), (img.shape[1], "w_out", ref["W_out"])):
            # an integer decided in floating point: equal unless the oracle sits at a rounding tie
            x = side * math.sqrt(max(ref["r"], 0.0)) / 28
            assert s[key] == exp or (_near_half(x) and abs(s[key] - exp) == 28), (name, b, key)
        p0 += n

    # --- condense: resample (device-read target size == explicit size; oracle within 1 LSB) -----
    got = hp.resized_images()
    sizes = [(s["h_out"], s["w_out"]) for s in stats]
    explicit = torch.zeros_like(hp.resized)
    pace.pace_apc_resample_to(hp.d["img"], hp.img_off, hp.H, hp.W, [z[0] for z in sizes], [z[1] for z in sizes],
                              explicit, hp.dst_off)
    flat = explicit.cpu().numpy()
    for b, (img, g, (ho, wo)) in enumerate(zip(wl.images, got, sizes)):
        o = hp.dst_off[b]
        np.testing.assert_array_equal(g, flat[o:o + ho * wo * 3].reshape(ho, wo, 3))
    out2 = torch.zeros_like(hp.resized)
    pace.pace_apc_resample_to(hp.d["img"], hp.img_off, hp.H, hp.W, [z[0] for z in oracle_sizes],
                              [z[1] for z in oracle_sizes], out2, hp.dst_off)
    flat2 = out2.cpu().numpy()
    for b, (img, (ho, wo)) in enumerate(zip(wl.images, oracle_sizes)):
        o = hp.dst_off[b]
        mine = flat2[o:o + ho * wo * 3].reshape(ho, wo, 3).astype(np.int32)
        assert np.abs(mine - O.apc_resample(img, ho, wo).astype(np.int32)).max() <= 1, (name, b)

    # --- extract: attention maps ----------------------------------------------------------------
    s_vis = hp.s_vis[: int(wl.cu_vis[-1])].cpu().numpy()
    s_vis_ref = oracle_vit(f64(wl.vit_q), f64(wl.vit_k), wl.cu_patches, 1 / math.sqrt(80), 4, pool=pool)
    assert_scores_close(s_vis, s_vis_ref, what=f"{name} S_vis_raw")
    s_llm = hp.s_llm[: int(wl.cu_vis[-1])].cpu().numpy()
    s_llm_ref = O.llm_text_visual_importance(f64(wl.llm_q), f64(wl.llm_k), wl.cu_q, wl.cu_vis, 1 / math.sqrt(128))
    assert_scores_close(s_llm, s_llm_ref, what=f"{name} S_llm_raw")
    for b in range(wl.B):
        v0, v1 = wl.cu_vis[b], wl.cu_vis[b + 1]
        assert s_vis[v0:v1].sum() == pytest.approx(wl.n_patches[b] * 16, rel=1e-4)
        assert s_llm[v0:v1].sum() == pytest.approx(wl.specs[b].tq * 28, rel=1e-4)

    # --- extract: fusion, top-K, gather ----------------------------------------------------------
    s_final = hp.s_final[: int(wl.cu_vis[-1])].cpu().numpy()
    weights = hp.weights[: wl.B].cpu().numpy()
    kept = hp.kept[: int(hp.cu_keep[-1])].cpu().numpy()
    ref = O.ddae_select(s_llm_ref, s_vis_ref, wl.cu_vis, hp.K)
    k0 = 0
    for b in range(wl.B):
        v0, v1 = int(wl.cu_vis[b]), int(wl.cu_vis[b + 1])
        assert_scores_close(s_final[v0:v1], ref["S_final"][v0:v1], atol_frac=2e-3, what=f"{name}[{b}] S_final")
        assert np.all(np.abs(weights[b] - ref["weights"][b]) <= 2e-3 * ref["weights"][b])
        assert_kept_matches(kept[k0:k0 + hp.K[b]], ref["S_final"][v0:v1], hp.K[b], offset=v0)
        k0 += hp.K[b]
    rows = hp.rows[: len(kept)].view(torch.int16).cpu().numpy()
    E = wl.embed.view(np.int16)
    np.testing.assert_array_equal(rows, E[kept])                   # a gather is a copy
    idx = torch.from_numpy(ref["kept"].astype(np.int32)).cuda()     # oracle's kept rows, gathered on the GPU
    rows_ref = pace.pace_gather(hp.d["embed"], idx).view(torch.int16).cpu().numpy()
    np.testing.assert_array_equal(rows_ref, O.gather_rows(E, ref["kept"]))


def test_img4k_budget_5_percent(pace):
    """The 4K workload's second budget (5 %): select on the oracle's own raw maps."""
    wl = synth.make_workload("img4k", seed=0, parts=("llm",))
    rng = np.random.default_rng(4)
    nv = wl.n_vis[0]
    s_llm = O.llm_text_visual_importance(f64(wl.llm_q), f64(wl.llm_k), wl.cu_q, wl.cu_vis, 1 / math.sqrt(128))
    s_vis = rng.lognormal(0, 1, nv) * 64      # a ViT-like positive map
    K = O.budget(nv, 0.05)
    assert K == 527
    sf, w, kept = pace.pace_ddae_select(torch.from_numpy(s_llm.astype(np.float32)).cuda(),
                                        torch.from_numpy(s_vis.astype(np.float32)).cuda(), wl.cu_vis,
                                        np.array([0, K], np.int32))
    ref = O.ddae_fuse(s_llm.astype(np.float32).astype(np.float64), s_vis.astype(np.float32).astype(np.float64))
    assert_scores_close(sf.cpu().numpy(), ref["S_final"], atol_frac=2e-3)
    assert_kept_matches(kept.cpu().numpy(), ref["S_final"], K)


@pytest.mark.parametrize("name", ["img1344", "ragged16"])
def test_step_from_host_matches_resident_step(pace, name):
    """Three steps from pinned host memory (alternating device input slots, the ViT row pass in
    query-row pieces behind the copies) give the same bits as one step on resident inputs."""
    from paper_2608_27206_gb300.hotpath import HotPath
    wl = synth.make_workload(name, seed=1)
    hp = HotPath(wl, "cuda")
    hp.step()
    torch.cuda.synchronize()
    names = ("stats", "dist", "s_vis", "s_llm", "s_final", "weights", "kept", "rows")
    want = {k: getattr(hp, k).clone() for k in names}
    pinned = {k: v.pin_memory() for k, v in hp.host.items()}
    out = {k: torch.empty(tuple(getattr(hp, k).shape), dtype=getattr(hp, k).dtype).pin_memory()
           for k in ("kept", "rows", "s_final", "stats")}
    for v in hp.d.values():            # the resident copies must not be what the steps read
        v.zero_()
    cs = torch.cuda.Stream()
    for _ in range(3):
        hp.step_from_host(pinned, out, cs)
    torch.cuda.synchronize()
    code, where = pace.pace_device_status(clear=True)
    assert code == 0, (code, where)
    for k, v in out.items():
        assert torch.equal(v, want[k].cpu()), k
    for k in names:
        assert torch.equal(getattr(hp, k), want[k]), k
