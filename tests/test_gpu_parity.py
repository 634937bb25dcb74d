"""CUDA path vs the CPU oracle, element by element, through the C ABI.

Integer/index results (routing, counts, grouped layout) must be bit-exact
when both sides route from the same fp32 logits; floating results must meet
max|gpu - oracle| / max|oracle| <= 2e-2 (bf16 data, fp32 accumulation).
"""
import os
import subprocess
import sys

import numpy as np
import pytest
import torch

from oracle import moe_oracle as O
from paper_2601_14327_gb300 import _lib as L
from paper_2601_14327_gb300 import layer

from gpu_helpers import (assert_close, case_inputs, dx_perm_ref, oracle_inputs, rel_err,
                         run_gpu_layer, to_np, topk_margin, unblock_ab)

pytestmark = pytest.mark.gpu


@pytest.fixture(autouse=True)
def _clean_device_error():
    L.moe_device_error(clear=True)
    yield
    assert L.moe_device_error(clear=True) == 0


def _route_only(T, E, k, z, mask=None):
    dev = "cuda"
    zt = torch.from_numpy(np.ascontiguousarray(z, np.float32)).to(dev)
    m = None if mask is None else torch.as_tensor(mask, dtype=torch.uint8).to(dev)
    idx = torch.empty(T, k, dtype=torch.int32, device=dev)
    g = torch.empty(T, k, dtype=torch.float32, device=dev)
    cnt = torch.empty(E, dtype=torch.int32, device=dev)
    lo = torch.empty(T, E, dtype=torch.float32, device=dev)
    L.moe_route(None, None, None, m, T, 8, E, k, zt, lo, idx, g, cnt)
    torch.cuda.synchronize()
    return idx.cpu().numpy(), g.cpu().numpy(), cnt.cpu().numpy(), lo.cpu().numpy()


@pytest.mark.parametrize("T,E,k,n_masked", [(1000, 64, 6, 10), (777, 16, 2, 0), (513, 128, 8, 7),
                                            (300, 171, 8, 20), (257, 256, 8, 85), (100, 8, 8, 0)])
def test_route_bit_exact_from_shared_logits(T, E, k, n_masked):
    rng = np.random.default_rng(T + E)
    z = rng.standard_normal((T, E)).astype(np.float32)
    mask = np.ones(E, np.uint8)
    mask[rng.permutation(E)[:n_masked]] = 0
    idx, g, cnt, lo = _route_only(T, E, k, z, mask)
    zm = O.apply_mask(z, mask)
    oidx, og = O.route_topk(zm, k)
    assert (idx == oidx).all()
    np.testing.assert_allclose(g, og, rtol=0, atol=2e-6)
    assert (cnt == O.expert_counts(oidx, E)).all()
    assert (lo == zm).all()


def test_route_ties_go_to_lower_index():
    T, E, k = 400, 32, 5
    rng = np.random.default_rng(3)
    z = rng.integers(-2, 2, size=(T, E)).astype(np.float32)  # many exact ties
    z[(z == 0) & (rng.random(z.shape) < 0.5)] = -0.0  # -0 ties with +0
    idx, g, cnt, _ = _route_only(T, E, k, z)
    oidx, og = O.route_topk(z, k)
    assert (idx == oidx).all()
    np.testing.assert_allclose(g, og, rtol=0, atol=2e-6)


@pytest.mark.parametrize("T,d,E", [(777, 512, 64), (300, 1024, 171), (129, 256, 256),
                                   # two 128-token tiles per CTA (97..192 experts), the second
                                   # one partly past T
                                   (1000, 384, 100), (2500, 7168, 171),
                                   # d not a multiple of the 64-wide k-block (zero-filled tail),
                                   # few experts (MMA N = 16), one token, the smallest d
                                   (333, 200, 13), (1, 72, 256), (64, 8, 5), (50, 136, 2)])
def test_route_logits_fp32(T, d, E):
    inp = case_inputs(T, d, E, 2, 128, seed=5)
    o = oracle_inputs(inp)
    dev = "cuda"
    b = layer.MoELayerBuffers(layer.LayerShape(T, d, E, 2, 128), dev, backward=False)
    layer.route(b, inp["x"].to(dev), inp["w_router"].to(dev), inp["bias"].to(dev), keep_logits=True)
    torch.cuda.synchronize()
    z = b.logits.cpu().numpy().astype(np.float64)
    ref = O.router_logits(o["x"], o["w_router"], o["bias"]).astype(np.float64)
    scale = np.abs(o["x"]) @ np.abs(o["w_router"]) + np.abs(o["bias"])[None, :]
    assert (np.abs(z - ref) <= 1e-5 * scale + 1e-30).all()
    # routing from the GPU logits: tokens with a clear top-k margin match exactly
    idx = b.topk_idx.cpu().numpy()
    oidx, _ = O.route_topk(ref.astype(np.float32), 2)
    clear = topk_margin(ref, 2) > 1e-4
    assert (idx[clear] == oidx[clear]).all()


@pytest.mark.parametrize("T,d,E,k", [(3000, 256, 64, 8), (777, 512, 171, 4), (129, 200, 256, 8),
                                     # two 128-feature tiles per CTA, the second one partly
                                     # past d
                                     (1000, 384, 120, 4),
                                     # tokens not a multiple of the 64-token k-block, d not a
                                     # multiple of the 128-feature tile, MMA N = 16, one token
                                     (333, 136, 13, 2), (1, 72, 5, 1), (64, 8, 2, 2),
                                     (4100, 1024, 16, 2)])
def test_route_bwd_against_oracle(T, d, E, k):
    """moe_route_bwd alone, from the same fp32 gates and d_gate as the oracle."""
    dev = "cuda"
    inp = case_inputs(T, d, E, k, 128, seed=11)
    gen = torch.Generator().manual_seed(T + d)
    z = torch.randn(T, E, generator=gen)
    idx = torch.argsort(z, dim=1, descending=True)[:, :k].to(torch.int32).contiguous()
    gate = torch.softmax(torch.gather(z, 1, idx.long()), dim=1).contiguous()
    dg = torch.randn(T, k, generator=gen).contiguous()
    x = inp["x"]
    dz_ref, dw_ref = O.router_backward(x.double().numpy(), idx.numpy(), gate.double().numpy(),
                                       dg.double().numpy(), E)
    ws_bytes = L.moe_workspace_size(T, d, E, k, 128)
    ws = torch.empty(ws_bytes, dtype=torch.uint8, device=dev)
    dl = torch.empty(T, k, dtype=torch.float32, device=dev)
    dw = torch.full((d, E), float("nan"), dtype=torch.float32, device=dev)
    L.moe_route_bwd(x.to(dev), idx.to(dev), gate.to(dev), dg.to(dev), T, d, E, k, dl, dw, ws,
                    ws_bytes)
    torch.cuda.synchronize()
    g64, dg64 = gate.double().numpy(), dg.double().numpy()
    # fp32 arithmetic on both terms of the softmax backward
    zscale = np.abs(g64) * (np.abs(dg64) + np.sum(np.abs(g64 * dg64), axis=1, keepdims=True))
    assert (np.abs(dl.cpu().numpy() - dz_ref) <= 2e-6 * zscale + 1e-30).all()
    # dZ carried exactly by three bf16 terms, products exact, fp32 accumulation over T
    dzs = np.zeros((T, E))
    np.put_along_axis(dzs, idx.numpy().astype(np.int64), zscale, axis=1)
    scale = np.abs(x.double().numpy()).T @ dzs
    got = dw.cpu().numpy().astype(np.float64)
    assert np.isfinite(got).all()
    assert (np.abs(got - dw_ref) <= 1e-5 * scale + 1e-30).all()
    unused = np.setdiff1d(np.arange(E), idx.numpy())
    assert (got[:, unused] == 0).all()


def test_load_stats_bit_exact_and_accumulate():
    T, k, E = 5000, 8, 200
    rng = np.random.default_rng(1)
    idx = rng.integers(0, E, size=(T, k)).astype(np.int32)
    ti = torch.from_numpy(idx).cuda()
    cnt = torch.empty(E, dtype=torch.int32, device="cuda")
    L.moe_load_stats(ti, T, k, E, cnt, accumulate=False)
    L.moe_load_stats(ti, T, k, E, cnt, accumulate=True)
    torch.cuda.synchronize()
    assert (cnt.cpu().numpy() == 2 * np.bincount(idx.reshape(-1), minlength=E)).all()


def test_load_stats_flags_bad_expert():
    idx = torch.tensor([[0, 1], [2, 9]], dtype=torch.int32, device="cuda")
    cnt = torch.empty(4, dtype=torch.int32, device="cuda")
    L.moe_load_stats(idx, 2, 2, 4, cnt)
    assert L.moe_device_error(clear=True) == 1  # MOE_DEV_BAD_EXPERT
    assert cnt.cpu().tolist() == [1, 1, 1, 0]


def test_route_flags_too_few_live_experts():
    z = np.zeros((4, 6), np.float32)
    mask = np.array([1, 0, 0, 0, 0, 1], np.uint8)
    _route_only(4, 6, 3, z, mask)
    assert L.moe_device_error(clear=True) == 2  # MOE_DEV_TOO_FEW_LIVE


def _permute(inp, idx, E, k, counts=None):
    T, d = inp["x"].shape
    R = L.moe_perm_rows_max(T, k, E)
    dev = "cuda"
    ws_bytes = L.moe_workspace_size(T, d, E, k, 128)
    ws = torch.empty(max(ws_bytes, 256), dtype=torch.uint8, device=dev)
    goff = torch.empty(E + 1, dtype=torch.int32, device=dev)
    gcnt = torch.empty(E, dtype=torch.int32, device=dev)
    row = torch.empty(T, k, dtype=torch.int32, device=dev)
    xp = torch.full((R, d), float("nan"), dtype=torch.bfloat16, device=dev)
    ct = None if counts is None else torch.as_tensor(counts, dtype=torch.int32).to(dev)
    L.moe_permute(inp["x"].to(dev), torch.from_numpy(np.ascontiguousarray(idx, np.int32)).to(dev), ct,
                  T, d, E, k, R, goff, gcnt, row, xp, ws, ws.numel())
    torch.cuda.synchronize()
    return goff.cpu().numpy(), gcnt.cpu().numpy(), row.cpu().numpy(), xp.cpu()


@pytest.mark.parametrize("T,d,E,k,bias", [(3000, 256, 64, 6, "zipf"), (4097, 128, 16, 2, "none"),
                                          (1000, 512, 128, 8, "loguniform")])
def test_permute_bit_exact(T, d, E, k, bias):
    inp = case_inputs(T, d, E, k, 128, bias=bias, seed=9)
    o = oracle_inputs(inp)
    oidx, _ = O.route_topk(O.router_logits(o["x"], o["w_router"], o["bias"]), k)
    goff, gcnt, row, xp = _permute(inp, oidx, E, k, counts=O.expert_counts(oidx, E))
    ooff, ocnt, orow = O.permutation(oidx, E, 128)
    assert (goff == ooff).all() and (gcnt == ocnt).all() and (row == orow).all()
    x = inp["x"]
    assert torch.equal(xp[torch.from_numpy(orow.reshape(-1))], x.repeat_interleave(k, dim=0))
    for e in range(E):
        pad = xp[ooff[e] + ocnt[e]:ooff[e + 1]]
        assert (pad.float() == 0).all()


def test_permute_all_tokens_one_expert_and_empty():
    T, d, E, k = 700, 128, 8, 1
    inp = case_inputs(T, d, E, k, 128, seed=2)
    idx = np.full((T, 1), 5, np.int32)
    goff, gcnt, row, xp = _permute(inp, idx, E, k)
    ooff, ocnt, orow = O.permutation(idx, E, 128)
    assert (goff == ooff).all() and (gcnt == ocnt).all() and (row == orow).all()
    # no tokens at all
    inp0 = case_inputs(1, d, E, k, 128, seed=2)
    inp0["x"] = inp0["x"][:0]
    goff, gcnt, row, xp = _permute(inp0, np.zeros((0, 1), np.int32), E, k)
    assert (goff == 0).all() and (gcnt == 0).all()


def test_permute_flags_count_mismatch():
    T, d, E, k = 300, 128, 8, 2
    inp = case_inputs(T, d, E, k, 128, seed=4)
    rng = np.random.default_rng(0)
    idx = rng.integers(0, E, size=(T, k)).astype(np.int32)
    bad = np.bincount(idx.reshape(-1), minlength=E)
    bad[0] += 1
    _permute(inp, idx, E, k, counts=bad)
    assert L.moe_device_error(clear=True) == 3  # MOE_DEV_COUNT_MISMATCH


LAYER_CASES = [
    # T, d, E, k, F, bias, n_masked
    (512, 256, 16, 2, 512, "none", 0),        # the tiny workload
    (300, 128, 1, 1, 128, "none", 0),         # one expert, k=1: a dense SwiGLU MLP; N=128 tiles,
                                              # a weight-gradient pair with one row block
    (1, 256, 4, 2, 256, "zipf", 0),           # a single token
    (1500, 384, 12, 4, 640, "zipf", 3),       # ragged groups, BN=128 paths, empty groups
    (700, 512, 8, 8, 256, "zipf", 0),         # k = number of experts
    (2100, 256, 32, 2, 384, "loguniform", 0), # volatile load, several empty experts
    (3000, 256, 256, 8, 256, "zipf", 40),     # the maximum expert count (schedule arrays full),
                                              # many light and empty experts
]


@pytest.mark.parametrize("T,d,E,k,F,bias,n_masked", LAYER_CASES)
def test_layer_fwd_bwd_against_oracle(T, d, E, k, F, bias, n_masked):
    inp = case_inputs(T, d, E, k, F, bias=bias, seed=T)
    o = oracle_inputs(inp)
    mask = None
    if n_masked:
        mask = np.ones(E, np.uint8)
        mask[np.random.default_rng(1).permutation(E)[:n_masked]] = 0
    z = O.router_logits(o["x"], o["w_router"], o["bias"])  # shared fp32 logits
    ref = O.moe_layer(o["x"], o["w_router"], o["bias"], mask, k, o["w_gate_up"], o["w_down"],
                      dy=o["dy"], logits32=z)
    b = run_gpu_layer(inp, E, k, mask=mask, logits_in=z)
    # integer parts: bit-exact
    assert (b.topk_idx.cpu().numpy() == ref["topk_idx"]).all()
    assert (b.counts.cpu().numpy() == ref["counts"]).all()
    assert (b.group_offsets.cpu().numpy() == ref["group_offsets"]).all()
    assert (b.group_counts.cpu().numpy() == ref["group_counts"]).all()
    row = b.row_of_assignment.cpu().numpy()
    assert (row == ref["row_of_assignment"]).all()
    # floating parts, per assignment through the grouped layout
    flat = row.reshape(-1)
    nrows = lambda a: a.reshape(T * k, -1)
    np.testing.assert_allclose(b.topk_gate.cpu().numpy(), ref["gates"], rtol=0, atol=2e-6)
    ab = unblock_ab(to_np(b.ab), F)
    assert_close("a", ab[flat][:, :F], nrows(ref["a"]))
    assert_close("b", ab[flat][:, F:], nrows(ref["b"]))
    assert_close("h", to_np(b.h)[flat], nrows(ref["h"]))
    assert_close("o", to_np(b.out_perm)[flat], nrows(ref["o"]))
    assert_close("y", to_np(b.y), ref["y"])
    assert_close("d_gate", b.d_gate.cpu().numpy(), ref["d_gate"])
    assert_close("dA", to_np(b.d_ab)[flat][:, :F], nrows(ref["dA"]))
    assert_close("dB", to_np(b.d_ab)[flat][:, F:], nrows(ref["dB"]))
    assert_close("dX", to_np(b.dx_perm)[flat], dx_perm_ref(ref, o["w_router"], T, k))
    assert_close("dw_down", to_np(b.dw_down), ref["dw_down"])
    assert_close("dw_gate_up", to_np(b.dw_gate_up), ref["dw_gate_up"])
    assert_close("d_logits", b.d_logits.cpu().numpy(), ref["d_logits"])
    assert_close("dw_router", b.dw_router.cpu().numpy(), ref["dw_router"])
    assert_close("dx", to_np(b.dx), ref["dx"])
    # experts without tokens get exactly zero weight gradients
    empty = np.nonzero(ref["counts"] == 0)[0]
    for e in empty:
        assert (to_np(b.dw_down[e]) == 0).all() and (to_np(b.dw_gate_up[e]) == 0).all()
        assert (b.dw_router[:, e].cpu().numpy() == 0).all()


def test_tiny_workload_end_to_end_gpu_logits():
    """The tiny workload with the router computed on the GPU (no shared logits)."""
    T, d, E, k, F = 512, 256, 16, 2, 512
    inp = case_inputs(T, d, E, k, F, bias="none", seed=1000)
    o = oracle_inputs(inp)
    ref = O.moe_layer(o["x"], o["w_router"], o["bias"], None, k, o["w_gate_up"], o["w_down"],
                      dy=o["dy"])
    b = run_gpu_layer(inp, E, k)
    idx = b.topk_idx.cpu().numpy()
    clear = topk_margin(ref["logits"], k) > 1e-4
    assert clear.mean() > 0.99
    assert (idx[clear] == ref["topk_idx"][clear]).all()
    y = to_np(b.y)
    assert rel_err(y[clear], ref["y"][clear]) <= 2e-2
    assert rel_err(to_np(b.dx)[clear], ref["dx"][clear]) <= 2e-2
    if clear.all():
        assert_close("dw_gate_up", to_np(b.dw_gate_up), ref["dw_gate_up"])
        assert_close("dw_down", to_np(b.dw_down), ref["dw_down"])
        assert_close("dw_router", b.dw_router.cpu().numpy(), ref["dw_router"])


def test_etn_history_recorded_on_device_drives_algorithm_1():
    """ETN[ITER, L, E] filled slot by slot by moe_load_stats from routings made
    on the GPU, then the host-side Algorithm 1 vs the oracle on the oracle's
    own routing of the same logits."""
    ITER, NL, T, E, k = 3, 4, 700, 32, 4
    rng = np.random.default_rng(21)
    etn = torch.zeros(ITER, NL, E, dtype=torch.int32, device="cuda")
    etn_ref = np.zeros((ITER, NL, E), np.int64)
    for it in range(ITER):
        for layer in range(NL):
            skew = np.log(rng.dirichlet(np.full(E, 0.3)) + 1e-9).astype(np.float32)
            z = (rng.standard_normal((T, E)).astype(np.float32) + skew[None, :])
            idx, _, _, _ = _route_only(T, E, k, z)
            L.moe_load_stats(torch.from_numpy(idx).cuda(), T, k, E, etn[it, layer])
            oidx, _ = O.route_topk(z, k)
            etn_ref[it, layer] = O.expert_counts(oidx, E)
    torch.cuda.synchronize()
    got = etn.cpu().numpy()
    assert (got == etn_ref).all()
    alphas = [O.layer_alpha(NL, l, 0.2, 0.4) for l in range(NL)]
    m, n = L.laep_prune_layers(got, T, k, alphas, 0.1)
    om, on = O.prune_layers(etn_ref, T, k, alphas, 0.1)
    assert (m == om).all() and (n == on).all()


def test_layer_all_tokens_to_one_expert():
    """A bias that sends every token to one expert: one group, seven empty ones."""
    T, d, E, k, F = 900, 256, 8, 1, 256
    inp = case_inputs(T, d, E, k, F, bias="none", seed=77)
    inp["bias"][3] = 30.0
    o = oracle_inputs(inp)
    z = O.router_logits(o["x"], o["w_router"], o["bias"])
    ref = O.moe_layer(o["x"], o["w_router"], o["bias"], None, k, o["w_gate_up"], o["w_down"],
                      dy=o["dy"], logits32=z)
    assert (ref["topk_idx"] == 3).all()
    b = run_gpu_layer(inp, E, k, logits_in=z)
    assert (b.topk_idx.cpu().numpy() == 3).all()
    assert_close("y", to_np(b.y), ref["y"])
    assert_close("dx", to_np(b.dx), ref["dx"])
    assert_close("dw_gate_up", to_np(b.dw_gate_up), ref["dw_gate_up"])
    assert_close("dw_down", to_np(b.dw_down), ref["dw_down"])
    for e in range(E):
        if e != 3:
            assert not b.dw_gate_up[e].any() and not b.dw_down[e].any()


def test_layer_without_tokens():
    """T = 0: nothing is routed; every weight gradient is exactly zero."""
    T, d, E, k, F = 0, 256, 4, 2, 256
    inp = case_inputs(1, d, E, k, F, seed=3)
    inp["x"] = inp["x"][:0].contiguous()
    inp["dy"] = inp["dy"][:0].contiguous()
    dev = "cuda"
    g = {n: v.to(dev) for n, v in inp.items()}
    b = layer.MoELayerBuffers(layer.LayerShape(T, d, E, k, F), dev)
    b.dw_gate_up.fill_(1.0)
    b.dw_down.fill_(1.0)
    b.dw_router.fill_(1.0)
    layer.forward(b, g["x"], g["w_router"], g["bias"], g["w_gate_up"], g["w_down"])
    layer.backward(b, g["dy"], g["w_router"], g["w_gate_up"], g["w_down"])
    torch.cuda.synchronize()
    assert (b.group_offsets.cpu() == 0).all()
    assert not b.dw_gate_up.any() and not b.dw_down.any() and not b.dw_router.any()


# ---------------------------------------------------------------- gathered dispatch

@pytest.mark.parametrize("T,E,k", [(3000, 64, 6), (1000, 128, 8), (257, 16, 2)])
def test_permute_map_bit_exact(T, E, k):
    """moe_permute_map: the grouped layout of the oracle, and the token of every row."""
    dev = "cuda"
    rng = np.random.default_rng(T)
    oidx = np.stack([rng.choice(E, size=k, replace=False) for _ in range(T)]).astype(np.int32)
    R = L.moe_perm_rows_max(T, k, E)
    ws_bytes = L.moe_workspace_size(T, 128, E, k, 128)
    ws = torch.empty(ws_bytes, dtype=torch.uint8, device=dev)
    goff = torch.empty(E + 1, dtype=torch.int32, device=dev)
    gcnt = torch.empty(E, dtype=torch.int32, device=dev)
    row = torch.empty(T, k, dtype=torch.int32, device=dev)
    tok = torch.full((R,), -7, dtype=torch.int32, device=dev)
    L.moe_permute_map(torch.from_numpy(oidx).to(dev), None, T, E, k, R, goff, gcnt, row, tok, ws,
                      ws_bytes)
    torch.cuda.synchronize()
    ooff, ocnt, orow = O.permutation(oidx, E, 128)
    assert (goff.cpu().numpy() == ooff).all() and (gcnt.cpu().numpy() == ocnt).all()
    assert (row.cpu().numpy() == orow).all()
    tk = tok.cpu().numpy()
    assert (tk[orow.reshape(-1)] == np.repeat(np.arange(T), k)).all()
    for e in range(E):
        assert (tk[ooff[e] + ocnt[e]:ooff[e + 1]] == 0).all()
    assert (tk[ooff[E]:] == -7).all()  # rows past the layout are not written


def _layer_both_ways(inp, E, k, mask=None):
    dev = "cuda"
    T, d = inp["x"].shape
    F = inp["w_down"].shape[2]
    g = {n: v.to(dev) for n, v in inp.items()}
    m = None if mask is None else torch.as_tensor(mask, dtype=torch.uint8).to(dev)
    out = []
    for gather in (False, True):
        b = layer.MoELayerBuffers(layer.LayerShape(T, d, E, k, F), dev, backward=True,
                                  gather=gather)
        layer.forward(b, g["x"], g["w_router"], g["bias"], g["w_gate_up"], g["w_down"], m)
        layer.backward(b, g["dy"], g["w_router"], g["w_gate_up"], g["w_down"])
        torch.cuda.synchronize()
        out.append(b)
    return out


@pytest.mark.parametrize("T,d,E,k,F,n_masked", [(1500, 256, 16, 4, 256, 0),
                                                (777, 384, 24, 8, 128, 5),
                                                (1, 128, 8, 2, 128, 0),
                                                (0, 128, 4, 2, 128, 0),
                                                (2048, 256, 8, 1, 384, 3)])
def test_gathered_layer_equals_materialized(T, d, E, k, F, n_masked):
    """The gathered dispatch (X_perm never written) gives the materialized path's results
    bit for bit: outputs, every gradient, and the saved activations on real rows."""
    inp = case_inputs(T, d, E, k, F, seed=T + 3)
    mask = None
    if n_masked:
        mask = np.ones(E, np.uint8)
        mask[np.random.default_rng(E).choice(E, n_masked, replace=False)] = 0
    a, b = _layer_both_ways(inp, E, k, mask)
    assert torch.equal(a.row_of_assignment, b.row_of_assignment)
    assert torch.equal(a.group_offsets, b.group_offsets)
    for name in ["y", "dx", "dw_gate_up", "dw_down", "dw_router", "d_logits", "d_gate"]:
        assert torch.equal(getattr(a, name), getattr(b, name)), name
    rows = a.row_of_assignment.reshape(-1).long()
    for name in ["h", "out_perm", "dx_perm"]:
        assert torch.equal(getattr(a, name)[rows], getattr(b, name)[rows]), name
    rr = rows.cpu().numpy()
    ua = unblock_ab(a.ab.view(torch.int16).cpu().numpy(), F)
    ub = unblock_ab(b.ab.view(torch.int16).cpu().numpy(), F)
    assert (ua[rr] == ub[rr]).all()


def test_one_sm_gemm_kernel_against_oracle():
    """The one-SM GEMM kernel (MOE_GEMM_1SM=1, kept for A/B measurements against the
    CTA-pair kernel) on layer cases; the variable is read once per process, so the
    cases run in a child process."""
    env = dict(os.environ, MOE_GEMM_1SM="1")
    script = os.path.join(os.path.dirname(os.path.abspath(__file__)), "gpu_one_sm_check.py")
    r = subprocess.run([sys.executable, script], env=env, capture_output=True, text=True,
                       timeout=900)
    assert r.returncode == 0, r.stdout[-2000:] + r.stderr[-4000:]


@pytest.mark.parametrize("T,d,E,k,F", [(1500, 384, 12, 4, 640), (3000, 256, 256, 8, 256)])
def test_router_term_in_dx_epilogue_equals_unpermute_sum_form(T, d, E, k, F):
    """The router's share of dx, added per grouped row in the dX GEMM's epilogue (the
    layer's default), against the same term added per token by moe_permute_bwd: both
    within the bf16 rounding of their sums, and both against the oracle."""
    inp = case_inputs(T, d, E, k, F, seed=T + 1)
    o = oracle_inputs(inp)
    z = O.router_logits(o["x"], o["w_router"], o["bias"])
    ref = O.moe_layer(o["x"], o["w_router"], o["bias"], None, k, o["w_gate_up"], o["w_down"],
                      dy=o["dy"], logits32=z)
    b = run_gpu_layer(inp, E, k, logits_in=z)
    fused_dx = to_np(b.dx)
    # recompute dX rows without the router term and sum them with moe_permute_bwd's
    R = b.shape.rows_cap
    g = {n: v.cuda() for n, v in inp.items()}
    L.moe_grouped_ffn_bwd_dgrad(b.d_out_perm, b.ab, b.group_offsets, E, d, F, R, g["w_gate_up"],
                                g["w_down"], None, None, None, None, T, k, None, b.d_ab,
                                b.dx_perm, b.ws, b.ws_bytes)
    flat = b.row_of_assignment.cpu().numpy().reshape(-1)
    assert_close("dX without the router term", to_np(b.dx_perm)[flat], ref["dX"].reshape(T * k, -1))
    dx2 = torch.empty_like(b.dx)
    L.moe_permute_bwd(b.dx_perm, b.row_of_assignment, b.topk_idx, b.d_logits, g["w_router"], T,
                      d, E, k, dx2, b.ws, b.ws_bytes)
    torch.cuda.synchronize()
    assert L.moe_device_error(clear=True) == 0
    unfused_dx = to_np(dx2)
    assert_close("dx (router term in the dX epilogue)", fused_dx, ref["dx"])
    assert_close("dx (router term in the unpermute-sum)", unfused_dx, ref["dx"])
    # the two differ only by where the bf16 roundings (unit roundoff u = 2^-9) fall: each
    # form rounds its k rows (dX_j + router_j, or dX_j alone) and its final sum, so
    # |fused - unfused| <= u * (sum_j |dX_j + router_j| + sum_j |dX_j| + 2 |dx|); the
    # oracle's rows stand in for the GPU's, with a factor 2 for their own error
    rows = dx_perm_ref(ref, o["w_router"], T, k).reshape(T, k, -1)
    scale = (np.abs(rows).sum(axis=1) + np.abs(ref["dX"]).sum(axis=1)
             + 2 * np.abs(ref["dx"]))
    assert (np.abs(fused_dx - unfused_dx) <= 2.0 ** -8 * scale + 1e-30).all()


@pytest.mark.parametrize("T,d,E,k,F", [(1500, 384, 12, 4, 640), (3000, 256, 256, 8, 256),
                                       (700, 512, 8, 8, 256)])
def test_gate_gradient_from_dh_epilogue(T, d, E, k, F):
    """d_gate from the dH GEMM's epilogue (the layer's default: sum over each grouped row of
    dH * H, H recomputed from the saved pre-activations, divided by the gate) against the
    oracle's <dy, o> and against moe_unpermute_combine_bwd's dot product with the stored O.
    Both carry the bf16 roundings of their inputs (O, or g*dy and W_down); they must agree
    within those, and the layer's routing gradient with them."""
    inp = case_inputs(T, d, E, k, F, seed=T + 3)
    o = oracle_inputs(inp)
    z = O.router_logits(o["x"], o["w_router"], o["bias"])
    ref = O.moe_layer(o["x"], o["w_router"], o["bias"], None, k, o["w_gate_up"], o["w_down"],
                      dy=o["dy"], logits32=z)
    b = run_gpu_layer(inp, E, k, logits_in=z)
    fused = b.d_gate.cpu().numpy().astype(np.float64)
    assert_close("d_gate (dH epilogue)", fused, ref["d_gate"])
    dg2 = torch.empty_like(b.d_gate)
    L.moe_unpermute_combine_bwd(inp["dy"].cuda(), b.out_perm, b.row_of_assignment, b.topk_gate,
                                b.group_offsets, b.group_counts, T, d, E, k, None, dg2)
    torch.cuda.synchronize()
    assert L.moe_device_error(clear=True) == 0
    direct = dg2.cpu().numpy().astype(np.float64)
    assert_close("d_gate (combine backward)", direct, ref["d_gate"])
    # |difference| within a few bf16 roundings of the terms of the dot product
    scale = np.einsum("td,tjd->tj", np.abs(o["dy"]), np.abs(ref["o"]))
    assert (np.abs(fused - direct) <= 2.0 ** -6 * scale + 1e-30).all()
    assert_close("d_logits", b.d_logits.cpu().numpy(), ref["d_logits"])


def test_dynamic_schedule_equals_fixed_stride(tmp_path):
    """The CTA pairs claim tiles from a shared counter, so which pair computes a tile
    changes from run to run, but not the tile's arithmetic: every output and gradient
    equals, bit for bit, the fixed-stride schedule (MOE_GEMM_STATIC=1, read once per
    process, so that half runs in a child process)."""
    import gpu_schedule_check as G
    path = str(tmp_path / "static.pt")
    env = dict(os.environ, MOE_GEMM_STATIC="1")
    script = os.path.join(os.path.dirname(os.path.abspath(__file__)), "gpu_schedule_check.py")
    r = subprocess.run([sys.executable, script, path], env=env, capture_output=True, text=True,
                       timeout=900)
    assert r.returncode == 0, r.stdout[-2000:] + r.stderr[-4000:]
    static = torch.load(path)
    for i, dyn in enumerate(G.run_cases()):
        for n in G.NAMES:
            assert torch.equal(dyn[n], static[i][n]), (G.SCHEDULE_CASES[i], n)


def test_row_block_split_equals_single_launch(tmp_path):
    """On 2^18 or more grouped rows the activation GEMMs are two launches: the CTA-pair
    kernel over whole pairs of 128-row blocks, then the one-SM kernel over each group's odd
    last block. Every output and gradient equals, bit for bit, the single CTA-pair launch
    (MOE_GEMM_SPLIT=0, read once per process, so that half runs in a child process): both
    kernels add the same products in the same order."""
    import gpu_split_check as G
    path = str(tmp_path / "single.pt")
    env = dict(os.environ, MOE_GEMM_SPLIT="0")
    script = os.path.join(os.path.dirname(os.path.abspath(__file__)), "gpu_split_check.py")
    r = subprocess.run([sys.executable, script, path], env=env, capture_output=True, text=True,
                       timeout=900)
    assert r.returncode == 0, r.stdout[-2000:] + r.stderr[-4000:]
    single = torch.load(path)
    for i, split in enumerate(G.run_cases()):
        assert split["odd_groups"] > 0, G.SPLIT_CASES[i]
        for n in G.NAMES:
            assert torch.equal(split[n], single[i][n]), (G.SPLIT_CASES[i], n)


def test_pruned_experts_weight_gradients_untouched():
    """Pruned experts (LAEP mask 0) get no tile and no store in the weight-gradient GEMMs:
    their gradient buffers keep what the caller left there. A live expert that received no
    token still gets exact zeros, and the live experts match the oracle."""
    T, d, E, k, F = 1200, 256, 10, 2, 384
    inp = case_inputs(T, d, E, k, F, seed=5)
    o = oracle_inputs(inp)
    mask = np.ones(E, np.uint8)
    mask[[1, 6]] = 0
    z = O.router_logits(o["x"], o["w_router"], o["bias"])
    z[:, 3] = -1e30  # live, never selected
    ref = O.moe_layer(o["x"], o["w_router"], o["bias"], mask, k, o["w_gate_up"], o["w_down"],
                      dy=o["dy"], logits32=z)
    assert ref["counts"][3] == 0 and (ref["counts"][[1, 6]] == 0).all()
    dev = "cuda"
    g = {n: v.to(dev) for n, v in inp.items()}
    m = torch.as_tensor(mask).to(dev)
    sentinel = 1.5
    for one_stream in (False, True):
        b = layer.MoELayerBuffers(layer.LayerShape(T, d, E, k, F), dev, backward=True)
        b.dw_gate_up.fill_(sentinel)
        b.dw_down.fill_(sentinel)
        layer.forward(b, g["x"], g["w_router"], g["bias"], g["w_gate_up"], g["w_down"], m,
                      torch.from_numpy(z).to(dev))
        layer.backward(b, g["dy"], g["w_router"], g["w_gate_up"], g["w_down"],
                       overlap=not one_stream, active_mask=m)
        torch.cuda.synchronize()
        assert L.moe_device_error(clear=True) == 0
        for e in (1, 6):
            assert (b.dw_gate_up[e] == sentinel).all() and (b.dw_down[e] == sentinel).all()
        assert not b.dw_gate_up[3].any() and not b.dw_down[3].any()
        live = np.nonzero(mask)[0]
        assert_close("dw_gate_up", to_np(b.dw_gate_up)[live], ref["dw_gate_up"][live])
        assert_close("dw_down", to_np(b.dw_down)[live], ref["dw_down"][live])
        assert_close("dx", to_np(b.dx), ref["dx"])


def test_bounded_wait_expires_and_reports():
    """A pipeline wait that nothing satisfies (an mbarrier no one arrives on) gives up
    after its limit: the kernel returns, the device error word reads
    MOE_DEV_WAIT_TIMEOUT (4), and the context keeps running the library's kernels."""
    import time
    assert L.moe_device_error(clear=True) == 0
    t0 = time.perf_counter()
    L.moe_selftest_wait_timeout(50_000_000)  # 50 ms
    code = L.moe_device_error(clear=True)    # synchronizes the device
    dt = time.perf_counter() - t0
    assert code == 4
    assert 0.045 <= dt < 5.0
    z = np.random.default_rng(3).standard_normal((300, 16)).astype(np.float32)
    idx, g, cnt, _ = _route_only(300, 16, 2, z)
    oidx, _ = O.route_topk(z, 2)
    assert (idx == oidx).all() and cnt.sum() == 600


def test_combine_bwd_halves_equal_fused():
    """moe_unpermute_combine_bwd with one output NULL computes that half alone: the
    d_out_perm half and the d_gate half equal the fused call bit for bit."""
    T, d, E, k = 1000, 512, 16, 4
    dev = "cuda"
    inp = case_inputs(T, d, E, k, 128, seed=21)
    b = layer.MoELayerBuffers(layer.LayerShape(T, d, E, k, 128), dev, backward=True)
    g = {n: v.to(dev) for n, v in inp.items()}
    layer.forward(b, g["x"], g["w_router"], g["bias"], g["w_gate_up"], g["w_down"])
    args = (g["dy"], b.out_perm, b.row_of_assignment, b.topk_gate, b.group_offsets,
            b.group_counts, T, d, E, k)
    dop_f = torch.full_like(b.d_out_perm, float("nan"))
    dg_f = torch.full_like(b.d_gate, float("nan"))
    L.moe_unpermute_combine_bwd(*args, dop_f, dg_f)
    dop_h = torch.full_like(b.d_out_perm, float("nan"))
    dg_h = torch.full_like(b.d_gate, float("nan"))
    L.moe_unpermute_combine_bwd(*args, dop_h, None)
    L.moe_unpermute_combine_bwd(*args, None, dg_h)
    torch.cuda.synchronize()
    used = int(b.group_offsets[E].item())
    assert torch.equal(dop_f[:used], dop_h[:used])
    assert torch.equal(dg_f, dg_h)
    with pytest.raises(L.MoEError):
        L.moe_unpermute_combine_bwd(*args, None, None)


def test_layer_is_deterministic_and_stream_layout_independent():
    """Every reduction runs in a fixed order (split partials, router partial sums, combine
    sums) and the only atomics are integer counts, so a step gives the same bits every
    time, and the two-stream backward gives the same bits as the one-stream one."""
    T, d, E, k, F = 2000, 256, 16, 4, 256
    dev = "cuda"
    inp = case_inputs(T, d, E, k, F, seed=77)
    g = {n: v.to(dev) for n, v in inp.items()}
    outs = []
    for overlap in (True, True, False):
        b = layer.MoELayerBuffers(layer.LayerShape(T, d, E, k, F), dev, backward=True)
        layer.forward(b, g["x"], g["w_router"], g["bias"], g["w_gate_up"], g["w_down"])
        layer.backward(b, g["dy"], g["w_router"], g["w_gate_up"], g["w_down"], overlap=overlap)
        torch.cuda.synchronize()
        outs.append(b)
    names = ["topk_idx", "topk_gate", "counts", "row_of_assignment", "y", "dx", "dw_gate_up",
             "dw_down", "dw_router", "d_logits"]
    for other in outs[1:]:
        for n in names:
            assert torch.equal(getattr(outs[0], n), getattr(other, n)), n


FUSED_COMBINE_CASES = [
    # T, d, E, k, F, bias, n_masked
    (512, 256, 16, 2, 512, "none", 0),
    (1, 256, 4, 2, 256, "zipf", 0),
    (1500, 384, 12, 4, 640, "zipf", 3),       # BN = 128 down GEMM, empty groups
    (700, 512, 8, 8, 256, "zipf", 0),
    (3000, 256, 256, 8, 256, "zipf", 40),
]


@pytest.mark.parametrize("T,d,E,k,F,bias,n_masked", FUSED_COMBINE_CASES)
def test_fused_combine_against_oracle_and_unfused(T, d, E, k, F, bias, n_masked):
    """Combine in the down GEMM's epilogue: y against the oracle, against the unfused
    path within its rounding, O and every gradient bit for bit as unfused."""
    inp = case_inputs(T, d, E, k, F, bias=bias, seed=T + 3)
    o = oracle_inputs(inp)
    mask = None
    if n_masked:
        mask = np.ones(E, np.uint8)
        mask[np.random.default_rng(2).permutation(E)[:n_masked]] = 0
    z = O.router_logits(o["x"], o["w_router"], o["bias"])
    ref = O.moe_layer(o["x"], o["w_router"], o["bias"], mask, k, o["w_gate_up"], o["w_down"],
                      logits32=z)
    b0 = run_gpu_layer(inp, E, k, mask=mask, logits_in=z)
    b1 = run_gpu_layer(inp, E, k, mask=mask, logits_in=z, fused_combine=True)
    b2 = run_gpu_layer(inp, E, k, mask=mask, logits_in=z, backward=False, fused_combine=True)
    assert b2.out_perm is None
    assert_close("y", to_np(b1.y), ref["y"])
    # the unfused combine sums gate * bf16(O) in fp32 and rounds once; the fused one sums
    # gate * O before O's bf16 rounding: at most u = 2^-8 (bf16's unit roundoff, 8-bit
    # significand) of sum |gate * O| apart, plus each side's final rounding (u of |y|) and
    # the fp32 sums' own error
    row = b0.row_of_assignment.cpu().numpy()
    g = b0.topk_gate.cpu().numpy().astype(np.float64)
    absgo = (np.abs(to_np(b0.out_perm).astype(np.float64))[row] * g[:, :, None]).sum(axis=1)
    y0 = to_np(b0.y).astype(np.float64)
    for b in (b1, b2):
        y = to_np(b.y).astype(np.float64)
        bound = 2.0 ** -8 * (absgo + np.abs(y0) + np.abs(y)) + 2.0 ** -20 * absgo + 1e-30
        assert (np.abs(y - y0) <= bound).all(), float(np.max(np.abs(y - y0) / bound))
    # same [A|B], H and O on every real row, same backward
    flat = torch.from_numpy(row.reshape(-1).astype(np.int64)).cuda()
    for name in ["h", "out_perm"]:
        assert torch.equal(getattr(b0, name)[flat], getattr(b1, name)[flat]), name
    assert torch.equal(b0.h[flat], b2.h[flat])
    assert (unblock_ab(to_np(b0.ab), F)[row.reshape(-1)] ==
            unblock_ab(to_np(b1.ab), F)[row.reshape(-1)]).all()
    for name in ["dx", "dw_gate_up", "dw_down", "dw_router", "d_logits", "d_gate"]:
        assert torch.equal(getattr(b0, name), getattr(b1, name)), name


def test_fused_combine_without_tokens():
    dev = "cuda"
    s = layer.LayerShape(0, 256, 8, 2, 256)
    b = layer.MoELayerBuffers(s, dev, backward=False, fused_combine=True)
    gen = torch.Generator(device=dev).manual_seed(3)
    wgu = (torch.randn(8, 512, 256, generator=gen, device=dev) * 0.02).to(torch.bfloat16)
    wd = (torch.randn(8, 256, 256, generator=gen, device=dev) * 0.02).to(torch.bfloat16)
    x = torch.empty(0, 256, dtype=torch.bfloat16, device=dev)
    w = torch.randn(256, 8, generator=gen, device=dev)
    layer.forward(b, x, w, None, wgu, wd)
    torch.cuda.synchronize()
    assert b.y.shape == (0, 256) and (b.counts == 0).all()



def test_graph_replay_of_the_step_equals_eager():
    """bench.py times replays of a CUDA graph of the whole step (both streams): the replay
    on new inputs gives the same bits as an eager step on those inputs."""
    T, d, E, k, F = 1500, 256, 16, 4, 256
    dev = "cuda"
    a = {n: v.to(dev) for n, v in case_inputs(T, d, E, k, F, seed=5).items()}
    c = {n: v.to(dev) for n, v in case_inputs(T, d, E, k, F, seed=6).items()}
    shape = layer.LayerShape(T, d, E, k, F)

    def step(b, x, dy):
        layer.forward(b, x, a["w_router"], a["bias"], a["w_gate_up"], a["w_down"])
        layer.backward(b, dy, a["w_router"], a["w_gate_up"], a["w_down"])

    bg = layer.MoELayerBuffers(shape, dev, backward=True)
    x_in, dy_in = a["x"].clone(), a["dy"].clone()
    step(bg, x_in, dy_in)  # eager warm-up (one-time setup outside the capture)
    torch.cuda.synchronize()
    graph = torch.cuda.CUDAGraph()
    with torch.cuda.graph(graph):
        step(bg, x_in, dy_in)
    x_in.copy_(c["x"])
    dy_in.copy_(c["dy"])
    graph.replay()
    torch.cuda.synchronize()
    be = layer.MoELayerBuffers(shape, dev, backward=True)
    step(be, c["x"], c["dy"])
    torch.cuda.synchronize()
    for n in ["topk_idx", "topk_gate", "counts", "row_of_assignment", "y", "dx", "dw_gate_up",
              "dw_down", "dw_router", "d_logits"]:
        assert torch.equal(getattr(bg, n), getattr(be, n)), n
