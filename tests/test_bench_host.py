"""Host-side logic of bench.py that needs no GPU: the key that ties a committed DRAM
capture to the code it measured, and the clock sampler's restriction to the timed
region."""
import os

import bench


def test_traffic_key_ignores_comments_not_code(tmp_path, monkeypatch):
    src = "paper_2601_14327_gb300/csrc/route.cu"
    text = open(os.path.join(bench.ROOT, src), encoding="utf-8").read()
    base = bench.sources_digest([src])
    monkeypatch.setattr(bench, "ROOT", str(tmp_path))
    os.makedirs(tmp_path / os.path.dirname(src))

    def digest_of(t):
        (tmp_path / src).write_text(t, encoding="utf-8")
        return bench.sources_digest([src])

    assert digest_of(text) == base
    # comment edits and re-indentation keep the key
    assert digest_of(text.replace("// ", "//  the ", 3)) == base
    assert digest_of("/* a new block\n comment */\n" + text) == base
    assert digest_of(text.replace("\n", "\n  ", 5)) == base
    # a code edit, or an edit inside a string literal, changes it
    assert digest_of(text.replace("kRtBM = 128", "kRtBM = 64", 1)) != base
    assert digest_of(text.replace('"moe_route: logits"', '"moe_route: logit"', 1)) != base


def test_clock_sampler_keeps_the_timed_region():
    c = bench.ClockSampler(0)
    row = "{sm},2070,{u},1000,Not Active,Not Active,Not Active,{cap}"
    c.lines = [(0.0, row.format(sm=2070, u=0, cap="Not Active")),      # idle, before
               (1.0, row.format(sm=1500, u=100, cap="Active")),        # timed region
               (1.1, row.format(sm=1520, u=100, cap="Active")),
               (1.2, row.format(sm=1480, u=30, cap="Active")),         # a lagging sample
               (3.0, row.format(sm=2070, u=0, cap="Not Active"))]      # idle, after
    c.t0, c.t1 = 0.5, 2.0

    class _Done:
        def terminate(self): pass
        def wait(self, timeout=None): pass

    class _Joined:
        def join(self, timeout=None): pass

    c.proc, c.thread = _Done(), _Joined()
    out = c.stop()
    assert out["samples"] == 3 and out["samples_under_load"] == 2
    assert out["sm_mhz"] == 1510 and out["sm_max_mhz"] == 2070
    assert out["reasons"] == ["sw_power_cap"]


def test_tensor_peak_follows_the_timed_region():
    peaks = {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0,
             "source": "measured"}
    p, name = bench.tensor_peak(peaks, 0.26)
    assert p == 1900.0 and "burst" in name
    p, name = bench.tensor_peak(peaks, 2.1)
    assert p == 1700.0 and "sustained" in name


def test_oracle_sample_on_routed_experts_equals_the_full_layer():
    """The bounded CPU-baseline sample keeps only the experts its tokens are routed to; the
    oracle on that subset must give these tokens the full layer's routing, outputs and
    gradients (the subset's weight gradients are the full layer's rows of those experts)."""
    import numpy as np
    import torch

    from oracle import moe_oracle as O
    from paper_2601_14327_gb300 import synth

    T, d, E, k, F = 48, 32, 12, 3, 16
    inp = synth.make_layer_inputs(T, d, E, k, F, bias="zipf", zipf_s=1.2, seed=7)
    mask = torch.ones(E, dtype=torch.uint8)
    mask[[1, 5]] = 0
    n = 5
    h, n_exp = bench.sample_inputs(inp, mask, k, n)
    full = O.moe_layer(inp["x"][:n].float().numpy(), inp["w_router"].numpy(),
                       inp["bias"].numpy(), mask.numpy(), k, inp["w_gate_up"].float().numpy(),
                       inp["w_down"].float().numpy(), dy=inp["dy"][:n].float().numpy())
    sub = O.moe_layer(h["x"], h["w_router"], h["bias"], h["mask"], k, h["w_gate_up"],
                      h["w_down"], dy=h["dy"])
    used = np.unique(full["topk_idx"])
    assert n_exp == used.size < E
    np.testing.assert_array_equal(used[sub["topk_idx"]], full["topk_idx"])
    for name in ("gates", "y", "dx", "d_gate", "d_logits"):
        np.testing.assert_array_equal(sub[name], full[name])
    np.testing.assert_array_equal(sub["dw_gate_up"], full["dw_gate_up"][used])
    np.testing.assert_array_equal(sub["dw_down"], full["dw_down"][used])
    np.testing.assert_array_equal(sub["dw_router"], full["dw_router"][:, used])
    assert not full["dw_gate_up"][np.setdiff1d(np.arange(E), used)].any()


def test_per_clock_fraction_discounts_the_clock_difference():
    peaks = {"bf16_tflops_sustained": 1575.5, "sustained_sm_mhz": 1342.0}
    # the same work per clock as the reference at a higher clock is 1.0, not above it
    assert bench.per_clock_frac(1575.5 * 1500 / 1342, 1500.0, peaks) == 1.0
    assert bench.per_clock_frac(1496.0, 1485.0, peaks) == round((1496 / 1485) / (1575.5 / 1342), 4)
    assert bench.per_clock_frac(1496.0, None, peaks) is None
    assert bench.per_clock_frac(1496.0, 1485.0, {"bf16_tflops_sustained": 1.0,
                                                "sustained_sm_mhz": None}) is None
