"""The C ABI library builds, loads and exports every entry point of include/pace.h.

Only host-side functions are called here (no GPU in this environment): status strings,
parameter defaults, the budget helper and the workspace size queries.
"""
import ctypes
import os
import re
import subprocess

import numpy as np
import pytest

from oracle import pace_oracle as O
from paper_2608_27206_gb300 import build as pace_build

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "pace.h")


@pytest.fixture(scope="module")
def libpace():
    path = pace_build.build()
    from paper_2608_27206_gb300 import pace
    assert os.path.samefile(path, pace.LIB_PATH)
    return pace


def declared_functions():
    text = open(HEADER).read()
    return sorted(set(re.findall(r"PACE_API\s+[\w\s\*]+?\b(pace_\w+)\s*\(", text)))


def test_header_declares_the_hot_path_calls():
    names = declared_functions()
    for fn in ("pace_apc_density", "pace_apc_resample", "pace_vit_attn_importance",
               "pace_llm_text_visual_importance", "pace_ddae_select", "pace_gather"):
        assert fn in names


def test_library_exports_every_declared_symbol(libpace):
    out = subprocess.run(["nm", "-D", "--defined-only", libpace.LIB_PATH], capture_output=True, text=True,
                         check=True).stdout
    exported = set(re.findall(r"\sT\s+(pace_\w+)", out))
    missing = [n for n in declared_functions() if n not in exported]
    assert not missing, missing
    lib = ctypes.CDLL(libpace.LIB_PATH)
    for n in declared_functions():
        assert getattr(lib, n) is not None


def test_status_strings(libpace):
    assert libpace.status_string(0) == "PACE_OK"
    assert libpace.status_string(2) == "PACE_ERR_UNSUPPORTED_ARCH"
    assert libpace.status_string(5) == "PACE_ERR_TIMEOUT"
    assert libpace.status_string(99) == "PACE_ERR_UNKNOWN"


def test_param_defaults_match_paper(libpace, golden):
    g = golden("paper_hyperparameters.txt")
    p = libpace.apc_params()
    assert p.alpha == pytest.approx(g["alpha"]) and p.gamma == pytest.approx(g["gamma"])
    assert p.tail_frac == pytest.approx(g["tail_frac"]) and p.align == g["merge_unit"]
    assert p.r_min == 0.0 and p.r_max == 1.0
    assert libpace.ddae_params().tau == pytest.approx(g["tau"])
    assert libpace.ddae_params().fusion == libpace.DDAE_ADAPTIVE


def test_budget_matches_oracle(libpace):
    rng = np.random.default_rng(0)
    for _ in range(2000):
        n = int(rng.integers(0, 50000))
        f = float(rng.choice([0.05, 0.1, 0.25, 0.2, 0.5, 1.0, 0.0, rng.uniform()]))
        assert libpace.pace_budget(n, f) == O.budget(n, f), (n, f)


def test_workspace_queries(libpace):
    h, w = [448, 2156], [448, 3836]
    ws = libpace.pace_apc_density_workspace_size(h, w)
    n = 32 * 32 + 154 * 274
    assert ws >= 2 * 589 * 8 + 2 * 4 * n
    cu = np.array([0, 1024, 1024 + 42196], dtype=np.int32)
    v = libpace.pace_vit_attn_importance_workspace_size(cu, 16)
    assert v >= 16 * 4 * (cu[-1]) + 16 * 4 * cu[-1]        # L rows + per-head partial maps
    l = libpace.pace_llm_text_visual_importance_workspace_size([0, 64], [0, 256], 28, 4)
    assert l >= 28 * 128 * 4 + 4 * 256 * 4
    assert libpace.pace_vit_attn_importance_workspace_size([0], 16) == 0
    # full-sequence S_llm: L rows cover the query set (padded to 256 rows), the part map the visual tokens
    for qs, nq in (("vision_text", 1000 - 14), ("text", 1000 - 14 - 576), ("last", 1)):
        s = libpace.pace_llm_sequence_importance_workspace_size([0, 1000], [14], [576], 28, 4, qs)
        assert s >= 28 * ((nq + 255) // 256 * 256) * 32 + 4 * 576 * 4, qs
    assert libpace.pace_llm_sequence_importance_workspace_size([0, 10], [8], [4], 28, 4, "text") == 0   # past the end
    assert libpace.pace_llm_sequence_importance_workspace_size([0, 10], [0], [4], 28, 4, 3) == 0        # bad query set


def test_budget_vanilla_matches_oracle(libpace):
    """B = p1 p2 relative to Vanilla, capped at the condensed token count (host helper)."""
    from oracle import pace_oracle as O
    rng = np.random.default_rng(9)
    for _ in range(2000):
        nv = int(rng.integers(0, 50000))
        nc = int(rng.integers(0, nv + 1))
        f = float(rng.choice([0.05, 0.1, 0.25, rng.uniform(0, 1.2)]))
        assert libpace.pace_budget_vanilla(nv, nc, f) == O.budget_vanilla(nv, nc, f)
    assert libpace.pace_budget_vanilla(10549, 2660, 0.10) == 1055 and libpace.pace_budget_vanilla(10549, 900, 0.10) == 900


def test_vit_chunk_rows_ends_on_pair_blocks(libpace):
    """Chunk ends for the split row pass: nondecreasing, the last at the total, every end an
    image boundary or a whole number of 256-row blocks into its image."""
    cu = np.array([0, 516, 520, 648, 1948, 2336, 4388], np.int32)
    for n in (1, 2, 3, 5, 8, 40):
        e = libpace.vit_chunk_rows(cu, n)
        assert len(e) == n and e[-1] == cu[-1] and np.all(np.diff(e) >= 0) and e[0] >= 0
        for x in e:
            b = int(np.searchsorted(cu, x, side="right")) - 1
            assert x in cu or (x - cu[b]) % 256 == 0
    assert list(libpace.vit_chunk_rows([0, 42196], 4)) == [10496, 20992, 31488, 42196]
