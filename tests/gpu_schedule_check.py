"""Child-process half of test_gpu_parity.py::test_dynamic_schedule_equals_fixed_stride:
runs the layer cases of SCHEDULE_CASES through the C ABI and saves every output and
gradient to the path given as the first argument. The parent runs the same cases with
the default (dynamic) tile schedule, this process with the variable the library reads
once per process (MOE_GEMM_STATIC=1: a fixed stride over the tile list)."""
import os
import sys

HERE = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, HERE)
sys.path.insert(0, os.path.dirname(HERE))

import torch  # noqa: E402

from gpu_helpers import case_inputs, run_gpu_layer  # noqa: E402

# T, d, E, k, F, bias: skewed loads (light and heavy groups in one list), BN = 128
# tiles (d = 384), the maximum expert count, and more tiles than CTA pairs many times over
SCHEDULE_CASES = [
    (4000, 256, 16, 4, 512, "zipf"),
    (1500, 384, 12, 4, 640, "loguniform"),
    (3000, 256, 256, 8, 256, "zipf"),
    (8192, 512, 64, 6, 512, "zipf"),
]
NAMES = ["y", "dx", "h", "out_perm", "d_ab", "dx_perm", "dw_gate_up", "dw_down", "dw_router"]
GROUPED = {"h", "out_perm", "d_ab", "dx_perm"}  # rows past group_offsets[E] are never written


def run_cases():
    out = []
    for T, d, E, k, F, bias in SCHEDULE_CASES:
        b = run_gpu_layer(case_inputs(T, d, E, k, F, bias=bias, seed=T + E), E, k)
        used = int(b.group_offsets[-1])
        out.append({n: (getattr(b, n)[:used] if n in GROUPED else getattr(b, n)).cpu()
                    for n in NAMES})
    return out


if __name__ == "__main__":
    assert os.environ.get("MOE_GEMM_STATIC") == "1"
    torch.save(run_cases(), sys.argv[1])
    print("fixed-stride schedule: saved")
