"""pace_apc_density_static: the density call for callers that cannot allocate device memory.

Some callers cannot hand the library a scratch buffer (for example a plugin inside a host
framework that owns all device allocations, or a latency-critical path where cudaMalloc is
not allowed).  pace_apc_density_static keeps its scratch in a static device array owned by
the library.  These tests check, through the C ABI, that two calls in a row give the same
results as pace_apc_density on the same inputs (so nothing stale survives between calls in
the shared array), and that oversize requests are rejected on the host.
This file is collected last on purpose; it initialises everything it needs itself.
"""
import numpy as np
import pytest
import torch

from paper_2608_27206_gb300 import synth
from tests.helpers import assert_scores_close

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


def _compare(P, got, ref):
    d_s, st_s = got
    d_w, st_w = ref
    assert_scores_close(d_s.cpu().numpy(), d_w.cpu().numpy(), atol_frac=2e-3, atol=1e-5, what="d_i")
    for a, b in zip(P.stats_dict(st_s), P.stats_dict(st_w)):
        for k in ("phi", "rho_g", "d_top", "rho_d", "rho", "r"):
            assert abs(a[k] - b[k]) <= 2e-3 * max(abs(b[k]), 1e-3) + 2e-6, (k, a[k], b[k])
        for k in ("n_patches", "k_tail", "h_out", "w_out"):
            assert a[k] == b[k], (k, a[k], b[k])


def test_static_density_matches_workspace_density_twice(pace):
    P = pace
    rng = np.random.default_rng(21)
    first = [synth.make_image(rng, 448, 448, 4, 4, 0.5), synth.make_image(rng, 616, 1232, 6, 3, 0.2)]
    second = [synth.make_image(rng, 1344, 1344, 8, 8, 0.3)]
    a, b = _inputs(first), _inputs(second)
    got_a = P.pace_apc_density_static(*a)       # two calls in a row through the C ABI
    got_b = P.pace_apc_density_static(*b)
    torch.cuda.synchronize()
    _compare(P, got_a, P.pace_apc_density(*a))
    _compare(P, got_b, P.pace_apc_density(*b))
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
