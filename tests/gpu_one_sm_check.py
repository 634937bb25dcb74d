"""Child-process check of the one-SM GEMM kernel (selected by MOE_GEMM_1SM=1, which
the library reads once per process): layer cases through the C ABI against the
oracle. Run by test_gpu_parity.py::test_one_sm_gemm_kernel_against_oracle."""
import os
import sys

HERE = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, HERE)
sys.path.insert(0, os.path.dirname(HERE))

import numpy as np  # noqa: E402

from oracle import moe_oracle as O  # noqa: E402
from gpu_helpers import (assert_close, case_inputs, dx_perm_ref, oracle_inputs,  # noqa: E402
                         run_gpu_layer, to_np, unblock_ab)


def check(T, d, E, k, F, n_masked):
    inp = case_inputs(T, d, E, k, F, seed=T)
    o = oracle_inputs(inp)
    mask = None
    if n_masked:
        mask = np.ones(E, np.uint8)
        mask[np.random.default_rng(1).permutation(E)[:n_masked]] = 0
    z = O.router_logits(o["x"], o["w_router"], o["bias"])
    ref = O.moe_layer(o["x"], o["w_router"], o["bias"], mask, k, o["w_gate_up"], o["w_down"],
                      dy=o["dy"], logits32=z)
    b = run_gpu_layer(inp, E, k, mask=mask, logits_in=z)
    row = b.row_of_assignment.cpu().numpy()
    assert (row == ref["row_of_assignment"]).all()
    flat = row.reshape(-1)
    nrows = lambda a: a.reshape(T * k, -1)
    ab = unblock_ab(to_np(b.ab), F)
    assert_close("a", ab[flat][:, :F], nrows(ref["a"]))
    assert_close("h", to_np(b.h)[flat], nrows(ref["h"]))
    assert_close("y", to_np(b.y), ref["y"])
    assert_close("dA", to_np(b.d_ab)[flat][:, :F], nrows(ref["dA"]))
    assert_close("dX", to_np(b.dx_perm)[flat], dx_perm_ref(ref, o["w_router"], T, k))
    assert_close("dw_down", to_np(b.dw_down), ref["dw_down"])
    assert_close("dw_gate_up", to_np(b.dw_gate_up), ref["dw_gate_up"])
    assert_close("dx", to_np(b.dx), ref["dx"])
    for e in np.nonzero(ref["counts"] == 0)[0]:
        assert (to_np(b.dw_down[e]) == 0).all() and (to_np(b.dw_gate_up[e]) == 0).all()


if __name__ == "__main__":
    assert os.environ.get("MOE_GEMM_1SM") == "1"
    check(1500, 384, 12, 4, 640, 3)  # ragged groups, N tiles of 128, empty experts
    check(700, 512, 8, 8, 256, 0)    # k = number of experts
    print("one-SM GEMM kernel: ok")
