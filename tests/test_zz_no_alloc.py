"""pace_apc_density_static: the density call for callers that cannot allocate device memory.

Some callers cannot hand the library a scratch buffer (for example a plugin inside a host
framework that owns all device allocations, or a latency-critical path where cudaMalloc is
not allowed).  pace_apc_density_static keeps its scratch in a static device array owned by
the library.  It runs the same kernels as pace_apc_density (deterministic fixed-point column
sums), so its results must be bit-identical to that call's on the same inputs.  These tests
check, through the C ABI:
  * two calls in a row, the second with more images than the first (so sums left over in the
    shared array from the first call would show), bit-equal to pace_apc_density, and one of
    them against the fp64 oracle;
  * a call exactly at both limits (PACE_APC_STATIC_MAX_IMAGES images holding
    PACE_APC_STATIC_MAX_PATCHES patches) is accepted and bit-equal to pace_apc_density;
  * oversize requests are rejected on the host.
This file is collected last on purpose; it initialises everything it needs itself.
"""
import numpy as np
import pytest
import torch

from oracle import pace_oracle as O
from paper_2608_27206_gb300 import synth
from tests.helpers import assert_distances_close

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def pace():
    from paper_2608_27206_gb300 import build
    build.build()
    from paper_2608_27206_gb300 import pace as P
    P.pace_init(0)
    return P


def _inputs(images):
    buf, off = synth.pack_images(images)
    return torch.from_numpy(buf).cuda(), off, [im.shape[0] for im in images], [im.shape[1] for im in images]


def _assert_identical(got, ref):
    """Static and workspace calls run the same deterministic kernels: every bit must agree."""
    d_s, st_s = got
    d_w, st_w = ref
    assert torch.equal(d_s, d_w), "d_i differ from pace_apc_density"
    assert torch.equal(st_s, st_w), "stats differ from pace_apc_density"


def _assert_matches_oracle(P, got, images):
    d, st = got
    d = d.cpu().numpy()
    p0 = 0
    for im, s in zip(images, P.stats_dict(st)):
        ref = O.apc_density(im)
        n = ref["N"]
        assert s["n_patches"] == n and s["k_tail"] == ref["k_tail"]
        assert_distances_close(d[p0:p0 + n], ref["d"], what="static d_i")
        for k in ("phi", "d_top", "rho_d", "rho", "r"):
            assert abs(s[k] - ref[k]) <= 2e-3 * max(abs(ref[k]), 1e-3) + 2e-6, (k, s[k], ref[k])
        p0 += n


def test_static_density_matches_workspace_density_twice(pace):
    P = pace
    rng = np.random.default_rng(21)
    first = [synth.make_image(rng, 448, 448, 4, 4, 0.5), synth.make_image(rng, 616, 1232, 6, 3, 0.2)]
    second = [synth.make_image(rng, 1344, 1344, 8, 8, 0.3), synth.make_image(rng, 252, 980, 5, 2, 0.6),
              synth.make_image(rng, 896, 448, 4, 4, 0.1)]
    a, b = _inputs(first), _inputs(second)
    got_a = P.pace_apc_density_static(*a)       # two calls in a row through the C ABI,
    got_b = P.pace_apc_density_static(*b)       # the second with more images than the first
    torch.cuda.synchronize()
    _assert_identical(got_a, P.pace_apc_density(*a))
    _assert_identical(got_b, P.pace_apc_density(*b))
    _assert_matches_oracle(P, got_a, first)
    code, where = P.pace_device_status(clear=True)
    assert code == 0, (code, where)


def test_static_density_at_the_limits(pace):
    """Exactly PACE_APC_STATIC_MAX_IMAGES images of 64 x 64 patches = PACE_APC_STATIC_MAX_PATCHES."""
    P = pace
    assert P.PACE_APC_STATIC_MAX_IMAGES * 64 * 64 == P.PACE_APC_STATIC_MAX_PATCHES
    rng = np.random.default_rng(22)
    imgs = [synth.make_image(rng, 896, 896, 4, 4, float(f)) for f in np.linspace(0.0, 0.9, P.PACE_APC_STATIC_MAX_IMAGES)]
    small = _inputs(imgs[:3])
    P.pace_apc_density_static(*small)           # a smaller call first leaves its sums in the array
    full = _inputs(imgs)
    got = P.pace_apc_density_static(*full)
    torch.cuda.synchronize()
    _assert_identical(got, P.pace_apc_density(*full))
    # two of the images against the oracle (Eq. 1 is summed over all 4096^2 pairs there)
    d, st = got
    sub = (d[15 * 4096:16 * 4096], st[15:16])
    _assert_matches_oracle(P, sub, imgs[15:16])
    _assert_matches_oracle(P, (d[:4096], st[:1]), imgs[:1])
    code, where = P.pace_device_status(clear=True)
    assert code == 0, (code, where)


def test_static_density_rejects_oversize_requests(pace):
    P = pace
    img = np.zeros((28, 28, 3), dtype=np.uint8)
    with pytest.raises(P.PaceError) as e:
        P.pace_apc_density_static(*_inputs([img] * (P.PACE_APC_STATIC_MAX_IMAGES + 1)))
    assert e.value.status == P.PACE_ERR_INVALID_ARG
    big = np.zeros((14 * 257, 14 * 256, 3), dtype=np.uint8)     # 65792 patches > 65536
    with pytest.raises(P.PaceError) as e:
        P.pace_apc_density_static(*_inputs([big]))
    assert e.value.status == P.PACE_ERR_INVALID_ARG
