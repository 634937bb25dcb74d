"""Parity at the five workloads' full sizes, in the launch configuration that
bench.py times (its Workload class: same inputs, same one-time LAEP prune,
same buffers and calls), on outputs the oracle can evaluate one by one:

- routing: the oracle routes every token from its own fp64 logits rounded to
  fp32; tokens whose gaps among the k+1 largest logits are all clear (> 1e-4)
  must get the same experts in the same order. Every other token (a near tie,
  where several top-k choices are correct) must get a valid top-k of the
  oracle's logits: each selected logit within the tolerance of the oracle's
  k-th largest, in descending order within the tolerance, and gates equal to
  the softmax of the oracle's logits over the GPU's choice. The LAEP mask must be
  the oracle's.
- y and dx of 256 tokens, every token of the lightest non-empty expert among
  them, evaluated by the oracle on the GPU's (valid) routing;
- the whole weight gradient of the lightest non-empty expert, and blocks of 128
  consecutive features (whole rows of dW_gate / dW_up, whole columns of
  dW_down) of the heaviest and the median expert, each from every assignment
  the GPU routed to that expert;
- pruned experts' weight gradients untouched, live experts without tokens
  exactly zero;
- the router gradient through a property that holds at any size: the softmax
  Jacobian makes every token's d_logits sum to zero, so the columns of
  dw_router sum to zero as well; and sampled feature rows of dw_router (plus
  every d_logits entry) against the oracle's router backward evaluated on the
  GPU's own routing, gates and d_gate.
"""
import numpy as np
import pytest
import torch

import bench
from oracle import moe_oracle as O
from paper_2601_14327_gb300 import _lib as L
from paper_2601_14327_gb300 import synth

pytestmark = pytest.mark.gpu
TOL = 2e-2
SENTINEL = 1.5


class _Experts:
    """Lazy fp64 view of per-expert weights (only the experts a check touches)."""

    def __init__(self, w, keep=12):
        self.w = w
        self.shape = tuple(w.shape)
        self.cache = {}
        self.keep = keep

    def __getitem__(self, key):
        e = key[0] if isinstance(key, tuple) else key
        e = int(e)
        if e not in self.cache:
            if len(self.cache) >= self.keep:
                self.cache.pop(next(iter(self.cache)))
            self.cache[e] = self.w[e].double().cpu().numpy()
        m = self.cache[e]
        return m[key[1:]] if isinstance(key, tuple) else m


def _rel(got, ref):
    den = np.max(np.abs(ref))
    return float(np.max(np.abs(np.asarray(got, np.float64) - ref)) / (den if den else 1.0))


@pytest.mark.parametrize("cfg_id", [0, 1, 2, 3, 4])
def test_full_size_sampled_parity(cfg_id):
    L.moe_device_error(clear=True)
    # the forward-only workloads run their backward too here (extra coverage at full size)
    wl = bench.Workload(cfg_id, "cuda", backward=True)
    wl.bufs.dw_gate_up.fill_(SENTINEL)  # pruned experts' gradients must keep it
    wl.bufs.dw_down.fill_(SENTINEL)
    wl.step()
    torch.cuda.synchronize()
    assert L.moe_device_error(clear=True) == 0
    c, s, b, inp = wl.cfg, wl.shape, wl.bufs, wl.inp
    T, d, E, k, F = s.T, s.d, s.E, s.k, s.F

    # ---- the oracle's own routing of every token (and its LAEP decision) ----
    x = inp["x"].float().cpu().numpy()
    wr = inp["w_router"].cpu().numpy()
    bias = inp["bias"].cpu().numpy()
    mask = None
    if c.prune_lowest:
        # the decision is taken on the full expert set before any compaction
        full = synth.make_layer_inputs(T, d, c.E, k, F, bias=c.bias, zipf_s=c.zipf_s,
                                       seed=synth.seed_for(cfg_id), device="cuda",
                                       with_weights=False, backward=False)
        z0 = O.router_logits(x, full["w_router"].cpu().numpy(), full["bias"].cpu().numpy())
        idx0, _ = O.route_topk(z0, k)
        m0, n0 = O.prune_mask_lowest(O.expert_counts(idx0, c.E), c.prune_lowest, k)
        assert n0 == wl.n_pruned
        if wl.mask is not None:
            assert (wl.mask.cpu().numpy() == m0).all(), "LAEP mask differs"
            mask = m0
        else:  # compacted: the kept experts, in order, are the live ones
            assert (wl.keep == np.nonzero(m0)[0]).all()
    z = O.router_logits(x, wr, bias, mask)
    oidx, ogates = O.route_topk(z, k)
    gidx = b.topk_idx.cpu().numpy()
    # the ordered top-k is unique where every gap among the k+1 largest logits is
    # clear; the top-k SET is unique where the k-th/(k+1)-th gap is clear
    zs = np.sort(z.astype(np.float64), axis=1)[:, ::-1][:, :k + 1]
    gaps = zs[:, :-1] - zs[:, 1:] if E > k else np.full((T, 1), np.inf)
    set_clear = gaps[:, -1] > 1e-4
    clear = gaps.min(axis=1) > 1e-4
    assert clear.mean() > 0.98 and set_clear.mean() > 0.99
    assert (gidx[clear] == oidx[clear]).all()
    assert (np.sort(gidx[set_clear], 1) == np.sort(oidx[set_clear], 1)).all()
    n_unclear = int((~set_clear).sum())
    gcnt = b.counts.cpu().numpy()
    ocnt = O.expert_counts(oidx, E)
    assert gcnt.sum() == T * k
    assert np.abs(gcnt - ocnt).sum() <= 2 * k * n_unclear
    if mask is not None:
        assert (gcnt[mask == 0] == 0).all()
    # grouped layout is consistent with the GPU's own routing, bit for bit
    goff, gcounts, grow = O.permutation(gidx, E, 128)
    assert (b.group_offsets.cpu().numpy() == goff).all()
    assert (b.row_of_assignment.cpu().numpy() == grow).all()

    # ---- near ties: the GPU's choice is a valid top-k of the oracle's logits ----
    ztol = 1e-4
    zg = np.take_along_axis(z.astype(np.float64), gidx.astype(np.int64), axis=1)
    kth = zs[:, k - 1]
    assert (zg >= kth[:, None] - ztol).all(), "a selected expert is not among the top k"
    assert (np.diff(zg, axis=1) <= ztol).all(), "selected experts out of order"
    srt = np.sort(gidx, axis=1)
    assert (srt[:, 1:] != srt[:, :-1]).all(), "an expert selected twice"
    if mask is not None:
        assert (mask[gidx] == 1).all()
    gz = zg - zg.max(axis=1, keepdims=True)
    g_ref = np.exp(gz) / np.exp(gz).sum(axis=1, keepdims=True)
    ggates = b.topk_gate.cpu().numpy()
    np.testing.assert_allclose(ggates, g_ref, rtol=0, atol=ztol)

    # ---- 256 tokens: y and dx on the GPU's routing ----
    wgu, wdn = _Experts(inp["w_gate_up"]), _Experts(inp["w_down"])
    rng = np.random.default_rng(cfg_id)
    live = np.nonzero(gcnt > 0)[0]
    order = live[np.argsort(gcnt[live], kind="stable")]
    lightest, heaviest, median = int(order[0]), int(order[-1]), int(order[len(order) // 2])
    light_toks = np.nonzero((gidx == lightest).any(axis=1))[0][:192]
    rest = np.setdiff1d(np.arange(T), light_toks)
    n_more = min(T, 256) - light_toks.size
    toks = np.sort(np.concatenate([light_toks, rng.choice(rest, size=n_more, replace=False)]))
    tt = torch.from_numpy(toks).cuda()
    dyv = inp["dy"][tt].float().cpu().numpy()
    y_ref, dx_ref, _, _ = O.tokens_forward_backward(x[toks], gidx[toks], g_ref[toks], dyv, wr,
                                                    wgu, wdn)
    assert _rel(b.y[tt].float().cpu().numpy(), y_ref) <= TOL
    assert _rel(b.dx[tt].float().cpu().numpy(), dx_ref) <= TOL

    # ---- weight gradients: the lightest expert whole, feature blocks of two others ----
    dy_all = inp["dy"]
    for e, block in ((lightest, None), (median, 128), (heaviest, 128)):
        t_e, j_e = np.nonzero(gidx == e)
        dy_rows = dy_all[torch.from_numpy(t_e).cuda()].float().cpu().numpy()
        if block is None:
            feats = np.arange(F)
        else:  # 128 consecutive features: one 128-row tile of dW_gate and of dW_up
            f0 = int(rng.integers(0, F // block)) * block
            feats = np.arange(f0, f0 + block)
        dwd, dwg, dwu = O.expert_weight_grad_columns(e, feats, x[t_e], dy_rows, g_ref[t_e, j_e],
                                                     wgu, wdn)
        f_t = torch.from_numpy(feats).cuda()
        g_dwd = b.dw_down[e][:, f_t].T.float().cpu().numpy()
        g_dwg = b.dw_gate_up[e][f_t].float().cpu().numpy()
        g_dwu = b.dw_gate_up[e][f_t + F].float().cpu().numpy()
        assert _rel(g_dwd, dwd) <= TOL, ("dw_down", e)
        assert _rel(g_dwg, dwg) <= TOL, ("dw_gate", e)
        assert _rel(g_dwu, dwu) <= TOL, ("dw_up", e)
    # pruned experts (a mask): not written; live experts without tokens: exactly zero
    for e in np.nonzero(gcnt == 0)[0]:
        e = int(e)
        if mask is not None and mask[e] == 0:
            assert (b.dw_down[e] == SENTINEL).all() and (b.dw_gate_up[e] == SENTINEL).all()
        else:
            assert not b.dw_down[e].any() and not b.dw_gate_up[e].any()
        assert not b.dw_router[:, e].any()

    # ---- router gradient: d_logits rows and dw_router columns sum to zero ----
    dl = b.d_logits.cpu().numpy().astype(np.float64)
    g = b.topk_gate.cpu().numpy().astype(np.float64)
    dg = b.d_gate.cpu().numpy().astype(np.float64)
    row_scale = (g * np.abs(dg)).sum(1) + np.abs((g * dg).sum(1))
    assert (np.abs(dl.sum(1)) <= 1e-5 * row_scale + 1e-30).all()
    dwr = b.dw_router.cpu().numpy().astype(np.float64)
    col_scale = np.abs(x).T @ np.abs(dl).sum(1)  # bound on |sum_e dw_router[i, e]|
    assert (np.abs(dwr.sum(1)) <= 1e-4 * col_scale + 1e-6).all()
    # sampled feature rows of dw_router against the oracle's router backward, from the
    # GPU's own routing, gates and d_gate (so only the arithmetic is compared): fp32
    # softmax backward and fp32 accumulation over T tokens
    feats = np.unique(np.concatenate([[0, d - 1], rng.choice(d, size=14, replace=False)]))
    dz_ref, dw_ref = O.router_backward(x[:, feats], gidx, g, dg, E)
    zscale = np.abs(g) * (np.abs(dg) + np.abs(g * dg).sum(1, keepdims=True))
    assert (np.abs(dl - dz_ref) <= 2e-6 * zscale + 1e-30).all()
    dzs = np.zeros((T, E))
    np.put_along_axis(dzs, gidx.astype(np.int64), zscale, axis=1)
    scale = np.abs(x[:, feats]).T @ dzs
    assert (np.abs(dwr[feats] - dw_ref) <= 1e-5 * scale + 1e-30).all()
    del wl
    torch.cuda.empty_cache()
