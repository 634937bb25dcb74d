"""Child-process half of test_gpu_parity.py::test_row_block_split_equals_single_launch:
runs the layer cases of SPLIT_CASES through the C ABI and saves every output and gradient
to the path given as the first argument. The parent runs the same cases with the default
launch plan (activation GEMMs on 2^18 or more grouped rows: the CTA-pair kernel over whole
pairs of 128-row blocks, then the one-SM kernel over each group's odd last block), this
process with the variable the library reads once per process (MOE_GEMM_SPLIT=0: one
CTA-pair launch that computes and drops the odd blocks' second halves)."""
import os
import sys

HERE = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, HERE)
sys.path.insert(0, os.path.dirname(HERE))

import torch  # noqa: E402

from gpu_helpers import case_inputs, run_gpu_layer  # noqa: E402

# T, d, E, k, F, bias: T*k + 128*E >= 2^18 grouped rows; skewed loads, so that many groups
# have an odd number of blocks, some only one; d = 384 gives N = 128 tiles in down and dX
SPLIT_CASES = [
    (32768, 256, 64, 8, 256, "zipf"),
    (32768, 384, 128, 8, 128, "loguniform"),
]
NAMES = ["y", "dx", "h", "out_perm", "d_ab", "dx_perm", "d_gate", "dw_gate_up", "dw_down",
         "dw_router"]
GROUPED = {"h", "out_perm", "d_ab", "dx_perm"}  # rows past group_offsets[E] are never written


def run_cases():
    out = []
    for T, d, E, k, F, bias in SPLIT_CASES:
        b = run_gpu_layer(case_inputs(T, d, E, k, F, bias=bias, seed=T + E + d), E, k)
        used = int(b.group_offsets[-1])
        rows = (b.group_offsets[1:] - b.group_offsets[:-1]).cpu()
        out.append({"odd_groups": int(((rows // 128) % 2 == 1).sum()),
                    **{n: (getattr(b, n)[:used] if n in GROUPED else getattr(b, n)).cpu()
                       for n in NAMES}})
    return out


if __name__ == "__main__":
    assert os.environ.get("MOE_GEMM_SPLIT") == "0"
    torch.save(run_cases(), sys.argv[1])
    print("single launch: saved")
