"""CPU oracle for the LAEP MoE expert-layer hot path.

TEST INFRASTRUCTURE ONLY. This module is the slow, plain reference the CUDA
path is checked against. Only the tests, the smoke check and the benchmark's
CPU-baseline leg may import it; the library never calls it and has no CPU
fallback.

Every function states the passage of the paper it follows (Yuan3.0 Ultra
technical report, arXiv 2601.14327). Floating point is fp64 except where the
method fixes fp32: the router logits are rounded to fp32 and the routing
decision (top-k) is taken on those fp32 values, as the fp32 router does.

Where the paper is silent the readings below are used (each is listed with
its reason in the design notes):
  R1  router: linear, fp32, fixed additive bias; pruned experts get logit -inf.
  R2  top-k order: logit descending, ties to the lower expert index.
  R3  gates: softmax over the k selected logits only (renormalised top-k).
  R4  expert FFN: SwiGLU with three matrices, h = silu(x Wg^T) * (x Wu^T),
      o = h Wd^T (three matrices per expert, Table A1 parameter counts).
  R5  dropless: every (token, slot) assignment is processed.
  R6  permuted layout: assignments grouped by expert, ordered by (token, slot)
      inside a group; each group starts at a multiple of `pad` rows.
  R7  Eq. 1-2 / Algorithm 1: strict '<', thresholds S*topK*beta and
      S*topK*alpha/E in fp64, experts visited in stable ascending count order.
  R8  count mode: prune the P smallest counts (Eq. 2's largest=False top-K).
  R9  at least k experts are always kept (the paper does not say; routing
      needs k live experts).
  R10 bias fixed, not trained (no bias gradient); masked experts get a zero
      router gradient.
  R11 Algorithm 1 over ITER iterations: the running load sum restarts for every
      (iteration, layer); Marker counts how often each expert (by id, not by
      sorted position) is flagged; the number pruned per layer is the mean
      flagged count over the iterations, rounded half up; experts are pruned in
      descending Marker order, ties to the lower total load over the
      iterations, then the lower id; only experts flagged at least once.
  R12 Layer-adaptive alpha: the first and the last floor(L/6) layers use the
      edge value (0.2 in the paper), the others the middle value (0.4).
  R13 Algorithm 2: ties in the descending sort go to the lower expert id, ties
      in argmin to the lower group; when the expert count is not a multiple of
      the group count the per-group capacity is rounded up (the listing would
      otherwise never place the remainder).
  R14 an expert without assignments gets a zero weight gradient here; this
      stands for a live expert (the kernels leave a pruned expert's dW alone).
  R15 d_gate is <dy, o> for every slot; the kernels report 0 where the fp32
      gate underflowed to 0, which no gradient downstream can see (the routing
      backward multiplies d_gate by its gate).
"""
from __future__ import annotations

import numpy as np

# ----------------------------------------------------------------------------
# Router (Sec. 3.2: E[i,j,l] = 1 iff token j is routed to expert i)
# ----------------------------------------------------------------------------


def router_logits(x, w_router, bias=None, active_mask=None):
    """z[t,e] = sum_i x[t,i] * W_r[i,e] + b[e], rounded to fp32 (reading R1).

    x: [T,d] (bf16 values as float), w_router: [d,E] fp32, bias: [E] or None,
    active_mask: [E] (nonzero = keep) or None. Returns fp32 [T,E]; pruned
    experts get -inf so they can never be selected (Sec. 4: pruned experts
    receive no tokens).
    """
    z = np.asarray(x, np.float64) @ np.asarray(w_router, np.float64)
    if bias is not None:
        z = z + np.asarray(bias, np.float64)[None, :]
    z = z.astype(np.float32)
    if active_mask is not None:
        z[:, np.asarray(active_mask) == 0] = -np.inf
    return z


def apply_mask(logits32, active_mask):
    z = np.array(logits32, np.float32, copy=True)
    if active_mask is not None:
        z[:, np.asarray(active_mask) == 0] = -np.inf
    return z


def route_topk(logits32, k):
    """Top-k experts per token and their gates (readings R2, R3).

    Selection is on the fp32 logits: descending value, ties to the lower expert
    index (a stable sort of -z keeps equal keys in index order). Gates are the
    softmax over the k selected logits, computed in fp64.
    Returns (topk_idx int32 [T,k], gates fp64 [T,k]).
    """
    z = np.asarray(logits32, np.float32)
    T, E = z.shape
    if not 1 <= k <= E:
        raise ValueError("k out of range")
    order = np.argsort(-z, axis=1, kind="stable")[:, :k]
    sel = np.take_along_axis(z, order, axis=1).astype(np.float64)
    if np.any(~np.isfinite(sel)):
        raise ValueError("fewer than k experts are active for some token")
    ex = np.exp(sel - sel[:, :1])
    gates = ex / ex.sum(axis=1, keepdims=True)
    return order.astype(np.int32), gates


def expert_counts(topk_idx, E):
    """Per-expert token number (the ETN of Algorithm 1 Step 1; Eq. 1 LHS)."""
    return np.bincount(np.asarray(topk_idx).reshape(-1), minlength=E).astype(np.int64)


# ----------------------------------------------------------------------------
# LAEP pruning decision (Sec. 3.2, Eq. 1-2, Algorithm 1)
# ----------------------------------------------------------------------------


def prune_mask_alpha_beta(counts, S, k, alpha, beta):
    """One histogram of Algorithm 1 (ITER = 1, one layer).

    Experts are visited in ascending order of load (stable: ties go to the
    lower index first). The running sum of visited loads is the cumulative
    load of Eq. 2. An expert is flagged when the running sum is below
    S*topK*beta AND its own load is below S*topK*alpha/E (E = experts before
    pruning, Eq. 1's N). Returns (active_mask uint8 [E], n_pruned).
    """
    counts = np.asarray(counts, np.int64)
    E = counts.shape[0]
    beta_thr = float(S) * float(k) * float(beta)
    alpha_thr = float(S) * float(k) * float(alpha) / float(E)
    order = np.argsort(counts, kind="stable")
    mask = np.ones(E, np.uint8)
    cum = 0
    n_pruned = 0
    for e in order:
        cum += int(counts[e])
        if cum < beta_thr and int(counts[e]) < alpha_thr:
            if E - n_pruned > k:  # reading R9
                mask[e] = 0
                n_pruned += 1
    return mask, n_pruned


def prune_mask_lowest(counts, P, k=1):
    """Prune the P least-loaded experts (reading R8; ties: lower index first)."""
    counts = np.asarray(counts, np.int64)
    E = counts.shape[0]
    P = int(min(max(P, 0), E - k))
    order = np.argsort(counts, kind="stable")
    mask = np.ones(E, np.uint8)
    mask[order[:P]] = 0
    return mask, P


# ----------------------------------------------------------------------------
# Dispatch layout (reading R6)
# ----------------------------------------------------------------------------


def permutation(topk_idx, E, pad=128):
    """Grouped layout of the T*k assignments.

    Group e holds the assignments routed to e, in (token, slot) order, and
    starts at group_offsets[e], a multiple of `pad`; group_offsets[E] is the
    total padded row count. Returns (group_offsets [E+1], group_counts [E],
    row_of_assignment [T,k]).
    """
    idx = np.asarray(topk_idx)
    T, k = idx.shape
    counts = expert_counts(idx, E)
    padded = ((counts + pad - 1) // pad) * pad
    offsets = np.zeros(E + 1, np.int64)
    offsets[1:] = np.cumsum(padded)
    row = np.empty((T, k), np.int64)
    fill = offsets[:-1].copy()
    for t in range(T):
        for j in range(k):
            e = idx[t, j]
            row[t, j] = fill[e]
            fill[e] += 1
    return offsets, counts, row


# ----------------------------------------------------------------------------
# Expert FFN and combine (reading R4; Table A1 fixes three matrices per expert)
# ----------------------------------------------------------------------------


def silu(a):
    return a / (1.0 + np.exp(-a))


def silu_grad(a):
    s = 1.0 / (1.0 + np.exp(-a))
    return s * (1.0 + a * (1.0 - s))


def _assignments_of(topk_idx, e):
    """(t, j) pairs routed to expert e, in (token, slot) order."""
    t, j = np.nonzero(np.asarray(topk_idx) == e)
    return t, j


def moe_forward(x, topk_idx, gates, w_gate_up, w_down):
    """Expert FFN per assignment and gate-weighted combine, fp64.

    For every assignment (t, j) with expert e = topk_idx[t,j]:
      a = x[t] Wg_e^T, b = x[t] Wu_e^T, h = silu(a) * b, o = h Wd_e^T,
    then y[t] = sum_j gates[t,j] * o[t,j].
    W_gate_up[e] stacks Wg_e (rows 0..F-1) over Wu_e (rows F..2F-1).
    Returns per-assignment a, b, h, o with shape [T,k,*] and y [T,d].
    """
    x = np.asarray(x, np.float64)
    T, d = x.shape
    k = topk_idx.shape[1]
    E, twoF, _ = w_gate_up.shape
    F = twoF // 2
    a = np.zeros((T, k, F))
    b = np.zeros((T, k, F))
    h = np.zeros((T, k, F))
    o = np.zeros((T, k, d))
    for e in range(E):
        t, j = _assignments_of(topk_idx, e)
        if t.size == 0:
            continue
        wg = np.asarray(w_gate_up[e, :F], np.float64)
        wu = np.asarray(w_gate_up[e, F:], np.float64)
        wd = np.asarray(w_down[e], np.float64)
        xe = x[t]
        ae = xe @ wg.T
        be = xe @ wu.T
        he = silu(ae) * be
        a[t, j], b[t, j], h[t, j] = ae, be, he
        o[t, j] = he @ wd.T
    y = np.einsum("tj,tjd->td", np.asarray(gates, np.float64), o)
    return {"a": a, "b": b, "h": h, "o": o, "y": y}


def moe_backward(dy, x, topk_idx, gates, w_router, w_gate_up, w_down, fwd):
    """Gradients of the layer for upstream gradient dy, fp64.

    combine:  d_o[t,j] = g[t,j] dy[t];  d_gate[t,j] = <dy[t], o[t,j]>
    expert:   dH = d_o Wd_e;  dA = dH * b * silu'(a);  dB = dH * silu(a)
              dX[t,j] = dA Wg_e + dB Wu_e
              dWd_e = sum d_o^T h;  dWg_e = sum dA^T x;  dWu_e = sum dB^T x
    router:   softmax over the selected k (reading R3):
              dz[t,j] = g_j (d_gate_j - sum_i g_i d_gate_i); zero elsewhere
              dW_r[:, e] = sum over assignments to e of dz * x[t]
    input:    dx[t] = sum_j dX[t,j] + sum_j dz[t,j] W_r[:, e_j]
    Experts that receive no token get exactly zero weight gradients.
    """
    dy = np.asarray(dy, np.float64)
    x = np.asarray(x, np.float64)
    g = np.asarray(gates, np.float64)
    T, d = x.shape
    k = topk_idx.shape[1]
    E, twoF, _ = w_gate_up.shape
    F = twoF // 2
    wr = np.asarray(w_router, np.float64)

    d_o = g[:, :, None] * dy[:, None, :]
    d_gate = np.einsum("td,tjd->tj", dy, fwd["o"])
    dA = np.zeros((T, k, F))
    dB = np.zeros((T, k, F))
    dX = np.zeros((T, k, d))
    dw_gate_up = np.zeros((E, twoF, d))
    dw_down = np.zeros((E, d, F))
    for e in range(E):
        t, j = _assignments_of(topk_idx, e)
        if t.size == 0:
            continue
        wg = np.asarray(w_gate_up[e, :F], np.float64)
        wu = np.asarray(w_gate_up[e, F:], np.float64)
        wd = np.asarray(w_down[e], np.float64)
        doe = d_o[t, j]
        ae, be, he = fwd["a"][t, j], fwd["b"][t, j], fwd["h"][t, j]
        dh = doe @ wd
        dae = dh * be * silu_grad(ae)
        dbe = dh * silu(ae)
        dA[t, j], dB[t, j] = dae, dbe
        dX[t, j] = dae @ wg + dbe @ wu
        xe = x[t]
        dw_down[e] = doe.T @ he
        dw_gate_up[e, :F] = dae.T @ xe
        dw_gate_up[e, F:] = dbe.T @ xe

    dz, dw_router = router_backward(x, topk_idx, g, d_gate, E)
    dx = dX.sum(axis=1) + np.einsum("tj,dtj->td", dz, wr[:, topk_idx])
    return {"d_o": d_o, "d_gate": d_gate, "dA": dA, "dB": dB, "dX": dX,
            "dw_gate_up": dw_gate_up, "dw_down": dw_down, "d_logits": dz,
            "dw_router": dw_router, "dx": dx}


def router_backward(x, topk_idx, gates, d_gate, E):
    """Router part of the backward, fp64: the softmax over the selected k
    (reading R3) and the linear router's weight gradient.

    dz[t,j] = g_j (d_gate_j - sum_i g_i d_gate_i)
    dW_r[:, e] = sum over assignments (t,j) to e of dz[t,j] x[t]  (zero if none)
    Returns (dz [T,k], dW_r [d,E]).
    """
    x = np.asarray(x, np.float64)
    g = np.asarray(gates, np.float64)
    d_gate = np.asarray(d_gate, np.float64)
    dz = g * (d_gate - np.sum(g * d_gate, axis=1, keepdims=True))
    dw_router = np.zeros((x.shape[1], E))
    for e in range(E):
        t, j = _assignments_of(topk_idx, e)
        if t.size:
            dw_router[:, e] = x[t].T @ dz[t, j]
    return dz, dw_router


def moe_layer(x, w_router, bias, active_mask, k, w_gate_up, w_down, dy=None,
              logits32=None, pad=128):
    """The whole hot path: route, count, permute, FFN, combine (and backward).

    If logits32 is given it replaces x W_r + b (the mask is still applied).
    """
    if logits32 is None:
        z = router_logits(x, w_router, bias, active_mask)
    else:
        z = apply_mask(logits32, active_mask)
    idx, gates = route_topk(z, k)
    E = w_gate_up.shape[0]
    counts = expert_counts(idx, E)
    offsets, gcounts, row = permutation(idx, E, pad)
    fwd = moe_forward(x, idx, gates, w_gate_up, w_down)
    out = {"logits": z, "topk_idx": idx, "gates": gates, "counts": counts,
           "group_offsets": offsets, "group_counts": gcounts,
           "row_of_assignment": row, **fwd}
    if dy is not None:
        out.update(moe_backward(dy, x, idx, gates, w_router, w_gate_up, w_down, fwd))
    return out


def to_permuted(per_assignment, row_of_assignment, n_rows):
    """Scatter a [T,k,*] per-assignment array into the grouped [n_rows,*] layout
    (pad rows are zero)."""
    pa = np.asarray(per_assignment)
    T, k = row_of_assignment.shape
    out = np.zeros((n_rows,) + pa.shape[2:], pa.dtype)
    out[np.asarray(row_of_assignment).reshape(-1)] = pa.reshape((T * k,) + pa.shape[2:])
    return out


# ----------------------------------------------------------------------------
# Per-element evaluation for large workloads: each value from its definition
# ----------------------------------------------------------------------------


def token_forward(x_t, experts, gates_t, w_gate_up, w_down):
    """y for a single token from its selected experts and gates (fp64)."""
    x_t = np.asarray(x_t, np.float64)
    F = w_gate_up.shape[1] // 2
    y = np.zeros_like(x_t)
    outs = []
    for e, g in zip(experts, gates_t):
        wgu = np.asarray(w_gate_up[e], np.float64)
        a = wgu[:F] @ x_t
        b = wgu[F:] @ x_t
        o = np.asarray(w_down[e], np.float64) @ (silu(a) * b)
        outs.append((a, b, o))
        y += g * o
    return y, outs


def token_backward(dy_t, x_t, experts, gates_t, w_router, w_gate_up, w_down):
    """dx and the router logit gradients for a single token (fp64)."""
    dy_t = np.asarray(dy_t, np.float64)
    x_t = np.asarray(x_t, np.float64)
    F = w_gate_up.shape[1] // 2
    g = np.asarray(gates_t, np.float64)
    _, outs = token_forward(x_t, experts, gates_t, w_gate_up, w_down)
    dgate = np.array([dy_t @ o for (_, _, o) in outs])
    dz = g * (dgate - np.sum(g * dgate))
    dx = np.zeros_like(x_t)
    for jj, (e, gj) in enumerate(zip(experts, g)):
        a, b, _ = outs[jj]
        wgu = np.asarray(w_gate_up[e], np.float64)
        dh = np.asarray(w_down[e], np.float64).T @ (gj * dy_t)
        da = dh * b * silu_grad(a)
        db = dh * silu(a)
        dx += wgu[:F].T @ da + wgu[F:].T @ db
        dx += dz[jj] * np.asarray(w_router, np.float64)[:, e]
    return dx, dgate, dz


def tokens_forward_backward(x_rows, experts, gates, dy_rows, w_router, w_gate_up, w_down):
    """y, dx, d_gate and d_logits of a set of tokens from their selected experts and gates
    (fp64): the definitions of token_forward / token_backward (and of moe_forward /
    moe_backward restricted to these tokens), evaluated expert by expert so that each
    expert's weights are read once for all the tokens routed to it.

    x_rows, dy_rows [n, d]; experts [n, k] (distinct per token); gates [n, k].
    Returns (y [n, d], dx [n, d], d_gate [n, k], d_logits [n, k]).
    """
    x = np.asarray(x_rows, np.float64)
    dy = np.asarray(dy_rows, np.float64)
    g = np.asarray(gates, np.float64)
    experts = np.asarray(experts)
    n, d = x.shape
    k = experts.shape[1]
    F = w_gate_up.shape[1] // 2
    o = np.zeros((n, k, d))
    dx = np.zeros((n, d))
    for e in np.unique(experts):
        t, j = np.nonzero(experts == e)  # each token at most once per expert
        wg = np.asarray(w_gate_up[e, :F], np.float64)
        wu = np.asarray(w_gate_up[e, F:], np.float64)
        wd = np.asarray(w_down[e], np.float64)
        xe = x[t]
        ae = xe @ wg.T
        be = xe @ wu.T
        o[t, j] = (silu(ae) * be) @ wd.T
        dh = (g[t, j][:, None] * dy[t]) @ wd
        dx[t] += (dh * be * silu_grad(ae)) @ wg + (dh * silu(ae)) @ wu
    y = np.einsum("tj,tjd->td", g, o)
    d_gate = np.einsum("td,tjd->tj", dy, o)
    dz = g * (d_gate - np.sum(g * d_gate, axis=1, keepdims=True))
    dx += np.einsum("tj,dtj->td", dz, np.asarray(w_router, np.float64)[:, experts])
    return y, dx, d_gate, dz


def expert_weight_grad_columns(e, feats, x_rows, dy_rows, gates_rows, w_gate_up, w_down):
    """Selected feature slices of expert e's weight gradients (fp64).

    x_rows, dy_rows, gates_rows: the token inputs, upstream gradients and gates
    of every assignment routed to e. For each feature f in `feats` returns
    dWd[:, f] (length d), dWg[f, :] and dWu[f, :] (length d) as arrays
    [len(feats), d]. The features are evaluated together: a, b, h and dH are
    [rows, len(feats)] matrices.
    """
    X = np.asarray(x_rows, np.float64)
    dY = np.asarray(dy_rows, np.float64)
    g = np.asarray(gates_rows, np.float64)
    F = w_gate_up.shape[1] // 2
    feats = np.asarray(feats)
    wd = np.asarray(w_down[e], np.float64)
    d_o = g[:, None] * dY
    a = X @ np.asarray(w_gate_up[e, feats], np.float64).T
    b = X @ np.asarray(w_gate_up[e, F + feats], np.float64).T
    h = silu(a) * b
    dh = d_o @ wd[:, feats]
    dwd = h.T @ d_o
    dwg = (dh * b * silu_grad(a)).T @ X
    dwu = (dh * silu(a)).T @ X
    return dwd, dwg, dwu


# ----------------------------------------------------------------------------
# Algorithm 1 over iterations and layers; the layer-adaptive alpha schedule
# ----------------------------------------------------------------------------


def layer_alpha(L, layer, alpha_edge=0.2, alpha_middle=0.4):
    """alpha of one layer (reading R12; Sec. 3.4.3 and the Table 5 caption)."""
    n6 = L // 6
    return alpha_edge if (layer < n6 or layer >= L - n6) else alpha_middle


def prune_layers(etn, S, k, alphas, beta):
    """Algorithm 1 with the ETN history of ITER iterations and L layers.

    etn: [ITER, L, E] per-expert token counts; alphas: [L]; returns
    (mask uint8 [L, E], n_pruned [L]) (reading R11).
    """
    etn = np.asarray(etn, np.int64)
    ITER, L, E = etn.shape
    marker = np.zeros((L, E), np.int64)
    exp_dis = np.zeros(L, np.int64)
    for it in range(ITER):
        for layer in range(L):
            counts = etn[it, layer]
            beta_thr = float(S) * float(k) * float(beta)
            alpha_thr = float(S) * float(k) * float(alphas[layer]) / float(E)
            order = np.argsort(counts, kind="stable")
            running = 0
            for e in order:
                running += int(counts[e])
                if running < beta_thr and int(counts[e]) < alpha_thr:
                    exp_dis[layer] += 1
                    marker[layer, e] += 1
    mask = np.ones((L, E), np.uint8)
    n_pruned = np.zeros(L, np.int64)
    total = etn.sum(axis=0)  # [L, E] load summed over the iterations
    for layer in range(L):
        n = (2 * int(exp_dis[layer]) + ITER) // (2 * ITER)
        n = min(n, E - k, int(np.count_nonzero(marker[layer])))
        ranked = sorted(range(E), key=lambda e: (-marker[layer, e], total[layer, e], e))
        for e in ranked[:n]:
            mask[layer, e] = 0
        n_pruned[layer] = n
    return mask, n_pruned


# ----------------------------------------------------------------------------
# Algorithm 2: expert rearrangement across n_g groups (devices)
# ----------------------------------------------------------------------------


def rearrange(loads, n_groups):
    """Greedy placement of experts into n_groups groups of equal size.

    Experts are taken in descending load order; each goes to the group with the
    smallest load sum that still has room (a full group is taken out of the
    argmin). Returns (order [n] = experts group by group, group_of [n],
    group_load [n_groups]) (reading R13).
    """
    loads = np.asarray(loads, np.int64)
    n = loads.shape[0]
    cap = -(-n // n_groups)  # == n // n_groups when n divides evenly
    order_desc = sorted(range(n), key=lambda e: (-loads[e], e))
    members = [[] for _ in range(n_groups)]
    sums = [0] * n_groups
    full = [False] * n_groups
    for e in order_desc:
        while True:
            g = min((g for g in range(n_groups)),
                    key=lambda g: (float("inf") if full[g] else sums[g], g))
            if len(members[g]) < cap:
                members[g].append(e)
                sums[g] += int(loads[e])
                break
            full[g] = True
    order = np.array([e for g in range(n_groups) for e in members[g]], np.int64)
    group_of = np.empty(n, np.int64)
    for g in range(n_groups):
        for e in members[g]:
            group_of[e] = g
    return order, group_of, np.array(sums, np.int64)

