"""C ABI checks that need no GPU: the library builds, loads and exports every
declared entry point; the host-side LAEP decision matches the oracle; argument
validation fails cleanly before any launch."""
import json
import os
import subprocess

import numpy as np
import pytest

from oracle import moe_oracle as O
from paper_2601_14327_gb300 import _lib as L
from paper_2601_14327_gb300 import build as B

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


@pytest.fixture(scope="module")
def lib():
    B.build()
    return L.load()


def test_library_exports_every_declared_symbol(lib):
    declared = L.header_functions()
    assert len(declared) >= 15
    out = subprocess.run(["nm", "-D", "--defined-only", B.LIB], capture_output=True, text=True,
                         check=True).stdout
    exported = {line.split()[-1] for line in out.splitlines() if line.strip()}
    missing = [f for f in declared if f not in exported]
    assert not missing, missing
    for f in declared:
        assert hasattr(lib, f)


def test_sizes(lib):
    assert L.moe_version() == 100
    assert L.moe_perm_rows_max(100, 8, 64) == 800 + 128 * 64
    ws = L.moe_workspace_size(16384, 4096, 64, 8, 2048)
    # router backward: dZ as three bf16 terms [3, 64, T] and the split partial sums of
    # dW_r [splits >= 1, d, 64]; transposed router [E, d]; partial logits [T, 64]; W_r
    # as three bf16 terms [3, 64, d]
    assert ws >= 3 * 64 * 16384 * 2 + 4096 * 64 * 4 + 64 * 4096 * 4 + 16384 * 64 * 4 \
        + 3 * 64 * 4096 * 2
    assert L.moe_workspace_size(0, 4096, 64, 8, 2048) >= 64 * 4096 * 4


def test_laep_prune_mask_golden(lib):
    g = json.load(open(os.path.join(GOLDEN, "laep_prune_cases.json")))
    for c in g["alpha_beta"]:
        mask, n = L.laep_prune_mask(c["counts"], c["S"], c["k"], c["alpha"], c["beta"], -1)
        assert mask == c["mask"] and n == c["n_pruned"], c["name"]
    for c in g["lowest"]:
        mask, n = L.laep_prune_mask(c["counts"], 1, c["k"], 0, 0, c["P"])
        assert mask == c["mask"] and n == c["n_pruned"], c["name"]


def test_laep_prune_mask_matches_oracle_random(lib):
    rng = np.random.default_rng(7)
    for _ in range(400):
        E = int(rng.integers(1, 257))
        k = int(rng.integers(1, min(E, 8) + 1))
        S = int(rng.integers(0, 5000))
        counts = rng.multinomial(S * k, rng.dirichlet(np.full(E, 0.2))) if S else np.zeros(E, int)
        alpha, beta = float(rng.uniform(0, 2)), float(rng.uniform(0, 0.5))
        m, n = L.laep_prune_mask(counts, S, k, alpha, beta, -1)
        om, on = O.prune_mask_alpha_beta(counts, S, k, alpha, beta)
        assert m == list(om) and n == on
        P = int(rng.integers(0, E + 1))
        m, n = L.laep_prune_mask(counts, S, k, 0, 0, P)
        om, on = O.prune_mask_lowest(counts, P, k)
        assert m == list(om) and n == on


def test_argument_validation_without_launch(lib):
    # E too large, k too large, d not a multiple of 128: rejected on the host
    with pytest.raises(L.MoEError) as e:
        L.moe_route(None, None, None, None, 10, 64, 300, 2, 1, None, 1, 1, None, None, 0, stream=0)
    assert e.value.status == -2
    with pytest.raises(L.MoEError) as e:
        L.moe_route(None, None, None, None, 10, 64, 16, 9, 1, None, 1, 1, None, None, 0, stream=0)
    assert e.value.status == -2
    with pytest.raises(L.MoEError) as e:
        L.moe_grouped_ffn_fwd(16, 16, 8, 100, 256, 4096, 16, 16, 16, 16, 16, 16, 0, stream=0)
    assert e.value.status == -2
    with pytest.raises(L.MoEError) as e:
        L.moe_grouped_ffn_fwd(None, 16, 8, 256, 256, 4096, 16, 16, 16, 16, 16, 16, 0, stream=0)
    assert e.value.status == -1
    # the grouped GEMMs need a workspace for their tile counter (16-byte aligned, 256 bytes)
    for ws, ws_bytes in ((None, 0), (16, 128), (24, 1 << 20)):
        with pytest.raises(L.MoEError) as e:
            L.moe_grouped_ffn_fwd(16, 16, 8, 256, 256, 4096, 16, 16, 16, 16, 16, ws, ws_bytes,
                                  stream=0)
        assert e.value.status == -6
        with pytest.raises(L.MoEError) as e:
            L.moe_grouped_ffn_bwd_dgrad(16, 16, 16, 8, 256, 256, 4096, 16, 16, None, None, None,
                                        None, 0, 1, None, 16, 16, ws, ws_bytes, stream=0)
        assert e.value.status == -6
        with pytest.raises(L.MoEError) as e:
            L.moe_grouped_ffn_bwd_wgrad(16, 16, 16, 16, 16, None, 8, 256, 256, 4096, 16, 16, ws,
                                        ws_bytes, stream=0)
        assert e.value.status == -6
    with pytest.raises(L.MoEError) as e:  # rows_cap below T*k + 128*E
        L.moe_permute(16, 16, None, 100, 64, 8, 2, 100, 16, 16, 16, 16, 16, 1 << 20, stream=0)
    assert e.value.status == -1
    with pytest.raises(L.MoEError) as e:  # workspace too small
        L.moe_permute(16, 16, None, 100, 64, 8, 2, 2000, 16, 16, 16, 16, 16, 8, stream=0)
    assert e.value.status == -6
    with pytest.raises(L.MoEError):
        L.laep_prune_mask([1, 2, 3], 2, 4)  # k > E


def test_laep_algorithms_golden(lib):
    g = json.load(open(os.path.join(GOLDEN, "laep_algorithms_cases.json")))
    for c in g["prune_layers"]:
        mask, n = L.laep_prune_layers(np.array(c["etn"]), c["S"], c["k"], c["alphas"], c["beta"])
        assert mask.tolist() == c["mask"] and n.tolist() == c["n_pruned"], c["name"]
    for c in g["layer_alpha"]:
        got = [L.laep_layer_alpha(c["L"], l) for l in range(c["L"])]
        if "alpha" in c:
            assert got == c["alpha"]
        else:
            assert sum(a == 0.2 for a in got) == c["edge_layers"]
    for c in g["rearrange"]:
        order, group_of, gl = L.laep_rearrange(c["loads"], c["n_groups"])
        assert order.tolist() == c["order"] and gl.tolist() == c["group_load"], c["name"]


def test_laep_algorithms_match_oracle_random(lib):
    rng = np.random.default_rng(11)
    for _ in range(150):
        E = int(rng.integers(2, 257))
        k = int(rng.integers(1, min(E, 8) + 1))
        iters, nl = int(rng.integers(1, 5)), int(rng.integers(1, 7))
        S = int(rng.integers(1, 3000))
        etn = np.stack([[rng.multinomial(S * k, rng.dirichlet(np.full(E, 0.25)))
                         for _ in range(nl)] for _ in range(iters)])
        alphas = [O.layer_alpha(nl, l, float(rng.uniform(0, 1)), float(rng.uniform(0, 1.5)))
                  for l in range(nl)]
        beta = float(rng.uniform(0, 0.4))
        m, n = L.laep_prune_layers(etn, S, k, alphas, beta)
        om, on = O.prune_layers(etn, S, k, alphas, beta)
        assert (m == om).all() and (n == on).all()
        ng = int(rng.integers(1, 9))
        loads = rng.integers(0, 10 ** 6, size=ng * int(rng.integers(1, 40)) + int(rng.integers(0, ng)))
        order, group_of, gl = L.laep_rearrange(loads, ng)
        oo, og, ogl = O.rearrange(loads, ng)
        assert (order == oo).all() and (group_of == og).all() and (gl == ogl).all()


def test_new_entry_points_validate_before_launch(lib):
    """Fused-dispatch entry points, the combine-backward halves and the wait self-test
    reject bad arguments on the host (no device work is queued)."""
    R = L.moe_perm_rows_max(100, 2, 8)
    with pytest.raises(L.MoEError) as e:  # no token_of_row
        L.moe_permute_map(16, None, 100, 8, 2, R, 16, 16, 16, None, 16, 1 << 20, stream=0)
    assert e.value.status == -1
    with pytest.raises(L.MoEError) as e:  # rows_cap below T*k + 128*E
        L.moe_permute_map(16, None, 100, 8, 2, 100, 16, 16, 16, 16, 16, 1 << 20, stream=0)
    assert e.value.status == -1
    with pytest.raises(L.MoEError) as e:  # workspace too small for the block histograms
        L.moe_permute_map(16, None, 100, 8, 2, R, 16, 16, 16, 16, 16, 4, stream=0)
    assert e.value.status == -6
    with pytest.raises(L.MoEError) as e:  # d not a multiple of 128
        L.moe_grouped_ffn_fwd_gather(16, 16, 10, 16, 8, 100, 256, R, 16, 16, 16, 16, 16, 16, 0,
                                     stream=0)
    assert e.value.status == -2
    with pytest.raises(L.MoEError) as e:  # x missing with tokens present
        L.moe_grouped_ffn_fwd_gather(None, 16, 10, 16, 8, 128, 256, R, 16, 16, 16, 16, 16, 16, 0,
                                     stream=0)
    assert e.value.status == -1
    with pytest.raises(L.MoEError) as e:  # unaligned token_of_row
        L.moe_grouped_ffn_bwd_wgrad_gather(16, 16, 20, 10, 16, 16, 16, None, 8, 128, 256, R, 16,
                                           16, 16, 1 << 20, stream=0)
    assert e.value.status == -1
    with pytest.raises(L.MoEError) as e:  # router backward: x missing with tokens present
        L.moe_route_bwd(None, 16, 16, 16, 10, 128, 8, 2, 16, 16, 16, 1 << 20, stream=0)
    assert e.value.status == -1
    with pytest.raises(L.MoEError) as e:  # router backward: unaligned x
        L.moe_route_bwd(24, 16, 16, 16, 10, 128, 8, 2, 16, 16, 16, 1 << 20, stream=0)
    assert e.value.status == -1
    with pytest.raises(L.MoEError) as e:  # router backward: k above E
        L.moe_route_bwd(16, 16, 16, 16, 10, 128, 4, 5, 16, 16, 16, 1 << 20, stream=0)
    assert e.value.status == -1
    with pytest.raises(L.MoEError) as e:  # router backward: workspace too small
        L.moe_route_bwd(16, 16, 16, 16, 10, 128, 8, 2, 16, 16, 16, 4, stream=0)
    assert e.value.status == -6
    Rf = L.moe_perm_rows_max(10, 2, 8)
    with pytest.raises(L.MoEError) as e:  # fused combine: k above E
        L.moe_grouped_ffn_fwd_combine(16, 16, 8, 128, 128, Rf, 16, 16, 16, 16, 10, 9, 16, 16,
                                      16, 16, 16, 16, 1 << 20, stream=0)
    assert e.value.status == -1
    with pytest.raises(L.MoEError) as e:  # fused combine: no y_acc with tokens present
        L.moe_grouped_ffn_fwd_combine(16, 16, 8, 128, 128, Rf, 16, 16, 16, 16, 10, 2, 16, 16,
                                      None, None, 16, 16, 1 << 20, stream=0)
    assert e.value.status == -1
    with pytest.raises(L.MoEError) as e:  # fused combine: rows_cap below T*k + 128*E
        L.moe_grouped_ffn_fwd_combine(16, 16, 8, 128, 128, 200, 16, 16, 16, 16, 10, 2, 16, 16,
                                      16, 16, 16, 16, 1 << 20, stream=0)
    assert e.value.status == -1
    with pytest.raises(L.MoEError) as e:  # fused combine: workspace too small
        L.moe_grouped_ffn_fwd_combine(16, 16, 8, 128, 128, Rf, 16, 16, 16, 16, 10, 2, 16, 16,
                                      16, 16, 16, 16, 4, stream=0)
    assert e.value.status == -6
    with pytest.raises(L.MoEError) as e:  # combine backward with neither output
        L.moe_unpermute_combine_bwd(16, 16, 16, 16, 16, 16, 10, 128, 8, 2, None, None, stream=0)
    assert e.value.status == -1
    with pytest.raises(L.MoEError) as e:  # router term: with tokens, every per-token input
        L.moe_grouped_ffn_bwd_dgrad(16, 16, 16, 8, 256, 256, 4096, 16, 16, 16, None, 16, 16, 10,
                                    2, None, 16, 16, 16, 1 << 20, stream=0)
    assert e.value.status == -1
    with pytest.raises(L.MoEError) as e:  # d_gate input without w_router
        L.moe_grouped_ffn_bwd_dgrad(16, 16, 16, 8, 256, 256, 4096, 16, 16, 16, 16, 16, None, 10,
                                    2, None, 16, 16, 16, 1 << 20, stream=0)
    assert e.value.status == -1
    with pytest.raises(L.MoEError) as e:  # d_gate both given and asked for
        L.moe_grouped_ffn_bwd_dgrad(16, 16, 16, 8, 256, 256, 4096, 16, 16, 16, 16, 16, 16, 10,
                                    2, 16, 16, 16, 16, 1 << 20, stream=0)
    assert e.value.status == -1
    with pytest.raises(L.MoEError) as e:  # gate gradient without row_of_assignment
        L.moe_grouped_ffn_bwd_dgrad(16, 16, 16, 8, 256, 256, 4096, 16, 16, 16, None, None, None,
                                    10, 2, 16, 16, 16, 16, 1 << 20, stream=0)
    assert e.value.status == -1
    with pytest.raises(L.MoEError) as e:  # router term: workspace for the per-row dz
        L.moe_grouped_ffn_bwd_dgrad(16, 16, 16, 8, 256, 256, 4096, 16, 16, 16, 16, 16, 16, 10,
                                    2, None, 16, 16, 16, 256, stream=0)
    assert e.value.status == -6
    for bad in (0, 999_999, 2_000_000_001):
        with pytest.raises(L.MoEError) as e:
            L.moe_selftest_wait_timeout(bad, stream=0)
        assert e.value.status == -1
