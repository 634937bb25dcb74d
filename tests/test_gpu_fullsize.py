"""Parity at the five workloads' full sizes, in the launch configuration that
bench.py times (its Workload class: same inputs, same one-time LAEP prune,
same buffers and calls), on outputs the oracle can evaluate one by one:

- routing: the oracle routes every token from its own fp64 logits rounded to
  fp32; tokens whose gaps among the k+1 largest logits are all clear (> 1e-4)
  must get the same experts in the same order, and tokens whose k-th/(k+1)-th
  gap is clear the same set; the histogram may differ only by the few
  near-tie tokens; the LAEP mask must be the same.
- y and dx of sampled tokens (token_forward / token_backward);
- selected feature slices of the weight gradients of sampled experts
  (heaviest, median, lightest non-empty) and exact zeros for empty experts;
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

    # ---- sampled tokens: y and dx ----
    wgu, wdn = _Experts(inp["w_gate_up"]), _Experts(inp["w_down"])
    rng = np.random.default_rng(cfg_id)
    cand = np.nonzero(clear)[0]
    toks = rng.choice(cand, size=min(12, cand.size), replace=False)
    y = b.y[torch.from_numpy(toks).cuda()].float().cpu().numpy()
    dx = b.dx[torch.from_numpy(toks).cuda()].float().cpu().numpy()
    dyv = inp["dy"][torch.from_numpy(toks).cuda()].float().cpu().numpy()
    ys, dxs = [], []
    for t, dyt in zip(toks, dyv):
        yt, _ = O.token_forward(x[t], oidx[t], ogates[t], wgu, wdn)
        dxt, _, _ = O.token_backward(dyt, x[t], oidx[t], ogates[t], wr, wgu, wdn)
        ys.append(yt)
        dxs.append(dxt)
    assert _rel(y, np.array(ys)) <= TOL
    assert _rel(dx, np.array(dxs)) <= TOL

    # ---- sampled experts: slices of the weight gradients ----
    live = np.nonzero(ocnt > 0)[0]
    order = live[np.argsort(ocnt[live], kind="stable")]
    experts = sorted({int(order[-1]), int(order[len(order) // 2]), int(order[0])})
    dy_all = inp["dy"]
    for e in experts:
        tt, jj = np.nonzero(oidx == e)
        feats = sorted(rng.choice(F, size=3, replace=False).tolist())
        dy_rows = dy_all[torch.from_numpy(tt).cuda()].float().cpu().numpy()
        dwd, dwg, dwu = O.expert_weight_grad_columns(e, feats, x[tt], dy_rows, ogates[tt, jj],
                                                     wgu, wdn)
        f_t = torch.tensor(feats).cuda()
        g_dwd = b.dw_down[e][:, f_t].T.float().cpu().numpy()
        g_dwg = b.dw_gate_up[e][f_t].float().cpu().numpy()
        g_dwu = b.dw_gate_up[e][f_t + F].float().cpu().numpy()
        assert _rel(g_dwd, dwd) <= TOL, ("dw_down", e)
        assert _rel(g_dwg, dwg) <= TOL, ("dw_gate", e)
        assert _rel(g_dwu, dwu) <= TOL, ("dw_up", e)
    empty = np.nonzero(gcnt == 0)[0]
    for e in empty[:4]:
        assert not b.dw_down[int(e)].any() and not b.dw_gate_up[int(e)].any()
        assert not b.dw_router[:, int(e)].any()

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
